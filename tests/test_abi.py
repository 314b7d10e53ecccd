"""The C-ABI library builds, loads without a GPU, and exports every declared symbol."""
import ctypes
import os

import pytest

from paper_2607_20791_gb300 import binding
from paper_2607_20791_gb300.build import build


@pytest.fixture(scope="module")
def lib_path():
    return build()


def test_header_declares_the_three_entry_points():
    syms = binding.header_symbols()
    for name in ("rgd_prefix_decode_attn", "rgd_sample_head", "rgd_probe_gate"):
        assert name in syms


def test_library_exports_every_header_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    missing = [s for s in binding.header_symbols() if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_covers_every_header_symbol():
    assert set(binding.header_symbols()) == set(binding._SIGNATURES)


def test_version_and_argument_errors_without_gpu(lib_path):
    lib = binding.load_library(lib_path)
    assert lib.rgd_version().decode().startswith("rgd")
    shape = binding.AttnShape(num_groups=1, rows_per_group=1, num_q_heads=4, num_kv_heads=1,
                              head_dim=96, page_size=16, num_pages=4, max_prompt_pages=1,
                              max_suffix_pages=1)
    assert lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(shape)) == 0
    assert b"head_dim" in lib.rgd_last_error_string()
    shape.head_dim = 128
    shape.num_ctas = 8
    assert lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(shape)) > 0
    # null pointers are rejected on the host before any launch
    rc = lib.rgd_sample_head(4, 100, 0, None, None, None, None, None, 0, None, None, None, None, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG
    rc = lib.rgd_probe_gate(None, 1, 1, None, 1, 1, -1, 4, None, None, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG
    # the residual precheck: theta outside [0, 1], a bad dtype, missing tensors
    for theta, dtype in ((1.5, 0), (-0.1, 0), (0.5, 7)):
        rc = lib.rgd_residual_precheck(4, 16, dtype, 1, 1, 0.0, theta, 5, None, 1, None, None, None)
        assert rc == binding.RGD_ERR_INVALID_ARG, (theta, dtype)
    assert b"theta" in lib.rgd_last_error_string() or b"dtype" in lib.rgd_last_error_string()
    rc = lib.rgd_residual_precheck(4, 16, 0, None, None, 0.0, 0.5, 5, None, None, None, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG
    assert lib.rgd_residual_precheck(0, 16, 0, None, None, 0.0, 0.5, 5, None, None, None, None, None) == 0
    # the soft gate: a NULL trie, top_k < 1
    rc = lib.rgd_soft_gate(None, 1, 1, 10, 0, None, 10, 5, 0.1, 2, -1, 8, None, None, None, None, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG
    # (the argument checks come before the trie is looked at: any non-NULL handle does here)
    rc = lib.rgd_soft_gate(1, 1, 1, 10, 0, 1, 10, 0, 0.1, 2, -1, 8, 1, None, 1, None, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG and b"top_k" in lib.rgd_last_error_string()


def test_gated_head_and_decode_step_argument_errors_without_gpu(lib_path):
    """The fused head + gate and the one-call step refuse bad arguments on the
    host, before any launch (the trie handle is not looked at before that)."""
    lib = binding.load_library(lib_path)
    P = 16  # any non-NULL, 16-byte aligned stand-in pointer
    args = lambda rows, rpg, max_len, trie=1, state=P: (rows, 100, 0, P, None, P, P, P, 0, None, P, None, trie,
                                                       rpg, -1, max_len, state, None, None)
    assert lib.rgd_sample_head_gated(*args(6, 4, 8)) == binding.RGD_ERR_INVALID_ARG  # 6 rows, groups of 4
    assert b"multiple" in lib.rgd_last_error_string()
    assert lib.rgd_sample_head_gated(*args(6, 3, 0)) == binding.RGD_ERR_INVALID_ARG  # max_len 0
    assert lib.rgd_sample_head_gated(*args(6, 3, 8, trie=None)) == binding.RGD_ERR_INVALID_ARG
    assert lib.rgd_sample_head_gated(*args(6, 256, 8)) == binding.RGD_ERR_INVALID_ARG  # rows_per_group > 255
    assert lib.rgd_sample_head_gated(*args(6, 3, 8, state=None)) == binding.RGD_ERR_INVALID_ARG
    assert lib.rgd_sample_head_gated(*args(6, 3, 8, state=P + 2)) == binding.RGD_ERR_INVALID_ARG  # misaligned
    assert lib.rgd_sample_head_gated(*args(0, 3, 8)) == 0  # an empty batch launches nothing
    shape = binding.AttnShape(num_groups=2, rows_per_group=3, num_q_heads=4, num_kv_heads=1, head_dim=128,
                              page_size=16, num_pages=4, max_prompt_pages=1, max_suffix_pages=1, num_ctas=4)
    # the head's arguments are checked first: max_len 0 is refused before the attention's
    rc = lib.rgd_decode_step(ctypes.byref(shape), P, P, P, P, P, P, P, 0.1, P, None, P, 1 << 20, 100, 0, P, None,
                             P, P, P, 0, None, P, None, 1, -1, 0, P, None, None)
    assert rc == binding.RGD_ERR_INVALID_ARG and b"max_len" in lib.rgd_last_error_string()
    assert lib.rgd_set_wait_limit_ns(0) == 0


def test_workspace_size_grows_with_blocks(lib_path):
    lib = binding.load_library(lib_path)
    s = binding.AttnShape(num_groups=16, rows_per_group=5, num_q_heads=32, num_kv_heads=8, head_dim=128,
                          page_size=16, num_pages=2000, max_prompt_pages=128, max_suffix_pages=16, num_ctas=100)
    a = lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(s))
    s.num_ctas = 400
    b = lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(s))
    # one ticket per job + (ctas + jobs - 1) partial slots of 20 queries x (128 + 2) floats
    grow = 300 * 20 * 128 * 4 + 300 * 20 * 8
    assert grow <= b - a < grow + 512  # each region is padded to 256 bytes
    s.reserved = 1
    assert lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(s)) == 0


def test_binding_refuses_undersized_tensors(lib_path):
    """The C side sees only pointers, so the binding checks every tensor's size
    against the shape before the call (CPU tensors reach that check before the
    device check, so this runs without a GPU)."""
    torch = pytest.importorskip("torch")
    binding.load_library(lib_path)
    shape = binding.AttnShape(num_groups=2, rows_per_group=3, num_q_heads=8, num_kv_heads=2, head_dim=64,
                              page_size=16, num_pages=10, max_prompt_pages=4, max_suffix_pages=2, num_ctas=4)
    R = 6
    bf, i32, u8, f32 = torch.bfloat16, torch.int32, torch.uint8, torch.float32
    good = dict(q=torch.empty(R * 8 * 64, dtype=bf), k_pages=torch.empty(10 * 2 * 16 * 64, dtype=bf),
                v_pages=torch.empty(10 * 2 * 16 * 64, dtype=bf), prompt_block_table=torch.empty(8, dtype=i32),
                prompt_len=torch.empty(2, dtype=i32), suffix_block_table=torch.empty(R * 2, dtype=i32),
                suffix_len=torch.empty(R, dtype=i32), row_active=torch.empty(R, dtype=u8), softmax_scale=0.125,
                out=torch.empty(R * 8 * 64, dtype=bf), lse=torch.empty(R * 8, dtype=f32))
    for name in ("q", "k_pages", "prompt_block_table", "prompt_len", "suffix_block_table", "suffix_len",
                 "row_active", "out", "lse"):
        args = dict(good)
        args[name] = good[name][:-1]
        with pytest.raises(ValueError, match=name):
            binding.rgd_prefix_decode_attn_noalloc(shape, **args)
    # with every size right, the next check is the device one
    with pytest.raises(ValueError, match="CUDA"):
        binding.rgd_prefix_decode_attn_noalloc(shape, **good)

    rows, vocab = 4, 50
    head = dict(logits=torch.empty(rows, vocab), is_probe=torch.empty(rows, dtype=u8),
                temperature=torch.empty(rows), min_p=torch.empty(rows), seed=torch.empty(rows, dtype=torch.int64),
                step=0, row_active=torch.empty(rows, dtype=u8), token_out=torch.empty(rows, dtype=i32),
                kept_count=torch.empty(rows, dtype=i32), kept_mask=torch.empty(rows * vocab, dtype=u8))
    for name in ("is_probe", "temperature", "min_p", "seed", "row_active", "token_out", "kept_count", "kept_mask"):
        args = dict(head)
        args[name] = head[name][:-1]
        with pytest.raises(ValueError, match=name):
            binding.rgd_sample_head(**args)

    class _NoTrie:
        handle = None
    st = torch.empty(3 * binding.GATE_STATE_BYTES - 1, dtype=u8)
    with pytest.raises(ValueError, match="state"):
        binding.rgd_gate_state_init(st, 3)
    with pytest.raises(ValueError, match="probe_tokens"):
        binding.rgd_probe_gate(_NoTrie(), 3, 2, torch.empty(2 * 5 + 3, dtype=i32), 4, 5, -1, 8, st)
    with pytest.raises(ValueError, match="logits"):
        binding.rgd_soft_gate(_NoTrie(), 3, 2, torch.empty(5 * 10 - 1), 20, 5, 0.1, 2, -1, 8, st,
                              torch.empty(3, dtype=i32))
    with pytest.raises(ValueError, match="w"):
        binding.rgd_residual_precheck(torch.empty(3, 16), torch.empty(15), 0.0, 0.5, 2, st)


def test_empty_batches_return_ok_without_a_launch(lib_path):
    """Zero rows or groups (or no tokens this call) is a valid call that does
    nothing; the pointers are not looked at."""
    lib = binding.load_library(lib_path)
    assert lib.rgd_sample_head(0, 100, 0, None, None, None, None, None, 0, None, None, None, None, None, None) == 0
    assert lib.rgd_gate_state_init(None, 0, None) == 0
    # (a non-NULL trie handle is required; it is not looked at for an empty call)
    assert lib.rgd_probe_gate(1, 0, 2, None, 1, 1, -1, 8, None, None, None, None) == 0
    assert lib.rgd_probe_gate(1, 4, 2, None, 0, 0, -1, 8, None, None, None, None) == 0
    assert lib.rgd_residual_precheck(0, 8, 1, None, None, 0.0, 0.5, 2, None, None, None, None, None) == 0
    # num_groups = 0 is an argument error for the attention call (its shape needs a group)
    shape = binding.AttnShape(num_groups=0, rows_per_group=1, num_q_heads=4, num_kv_heads=1, head_dim=128,
                              page_size=16, num_pages=1, max_prompt_pages=1, max_suffix_pages=1)
    assert lib.rgd_prefix_decode_attn_workspace_size(ctypes.byref(shape)) == 0
