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
