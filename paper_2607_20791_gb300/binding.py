"""Thin ctypes binding of the C ABI in ``include/rgd.h`` (argument marshalling only).

Every function here has the name of the C entry point it calls and does nothing
but check and convert arguments: torch CUDA tensors become device pointers, the
current torch CUDA stream becomes the stream argument, and a non-zero status is
raised as :class:`RgdError`.  All computation happens in the CUDA kernels of
``librgd.so``; there is no fallback.  If the library has not been built the first
call raises.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "librgd.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "rgd.h")

RGD_OK, RGD_ERR_INVALID_ARG, RGD_ERR_CUDA, RGD_ERR_UNSUPPORTED = 0, 1, 2, 3
RGD_DEV_BAD_PAGE, RGD_DEV_BAD_TOKEN, RGD_DEV_WAIT_TIMEOUT, RGD_DEV_BAD_PARAM = 1, 2, 4, 8
RGD_F32, RGD_BF16 = 0, 1
RGD_PENDING, RGD_REFUSAL, RGD_NON_REFUSAL = 0, 1, 2


class RgdError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"rgd error {code}: {msg}")
        self.code = code


class AttnShape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "num_groups", "rows_per_group", "num_q_heads", "num_kv_heads", "head_dim", "page_size",
        "num_pages", "max_prompt_pages", "max_suffix_pages", "num_ctas", "reserved")]


class GateState(ctypes.Structure):
    _fields_ = [("node", ctypes.c_int32), ("length", ctypes.c_int32), ("steps", ctypes.c_int32),
                ("decisive_step", ctypes.c_int32), ("decision", ctypes.c_uint8),
                ("confirmed", ctypes.c_uint8), ("done", ctypes.c_uint8), ("reserved", ctypes.c_uint8)]


GATE_STATE_BYTES = ctypes.sizeof(GateState)  # 20

_lib = None
_P = ctypes.c_void_p
_I32, _I64, _U64, _SZ, _F = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_size_t, ctypes.c_float

_SIGNATURES = {
    "rgd_last_error_string": (ctypes.c_char_p, []),
    "rgd_version": (ctypes.c_char_p, []),
    "rgd_set_wait_limit_ns": (ctypes.c_int, [_U64]),
    "rgd_prefix_decode_attn_workspace_size": (_SZ, [ctypes.POINTER(AttnShape)]),
    "rgd_prefix_decode_attn": (ctypes.c_int, [ctypes.POINTER(AttnShape), _P, _P, _P, _P, _P, _P, _P, _P, _F,
                                               _P, _P, _P, _SZ, _P, _P]),
    "rgd_prefix_decode_attn_noalloc": (ctypes.c_int, [ctypes.POINTER(AttnShape), _P, _P, _P, _P, _P, _P, _P,
                                                       _P, _F, _P, _P, _P, _P]),
    "rgd_sample_head": (ctypes.c_int, [_I32, _I32, _I32, _P, _P, _P, _P, _P, _U64, _P, _P, _P, _P, _P, _P]),
    "rgd_sample_head_gated": (ctypes.c_int, [_I32, _I32, _I32, _P, _P, _P, _P, _P, _U64, _P, _P, _P, _P, _I32,
                                             _I32, _I32, _P, _P, _P]),
    "rgd_decode_step": (ctypes.c_int, [ctypes.POINTER(AttnShape), _P, _P, _P, _P, _P, _P, _P, _F, _P, _P, _P,
                                       _SZ, _I32, _I32, _P, _P, _P, _P, _P, _U64, _P, _P, _P, _P, _I32, _I32,
                                       _P, _P, _P]),
    "rgd_trie_create": (ctypes.c_int, [_P, _P, _I32, _I32, ctypes.POINTER(_P)]),
    "rgd_trie_destroy": (ctypes.c_int, [_P]),
    "rgd_trie_info": (ctypes.c_int, [_P, ctypes.POINTER(_I32), ctypes.POINTER(_I32)]),
    "rgd_gate_state_init": (ctypes.c_int, [_P, _I32, _P]),
    "rgd_probe_gate": (ctypes.c_int, [_P, _I32, _I32, _P, _I32, _I64, _I32, _I32, _P, _P, _P, _P]),
    "rgd_residual_precheck": (ctypes.c_int, [_I32, _I32, _I32, _P, _P, _F, _F, _I32, _P, _P, _P, _P, _P]),
    "rgd_soft_gate": (ctypes.c_int, [_P, _I32, _I32, _I32, _I32, _P, _I64, _I32, _F, _I32, _I32, _I32, _P, _P,
                                     _P, _P, _P, _P]),
}


def header_symbols(path: str = HEADER):
    """Function names declared in the C header."""
    text = open(path).read()
    return sorted(set(re.findall(r"^\s*(?:[A-Za-z_][\w\s\*]*?)\b(rgd_\w+)\s*\(", text, re.M)))


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load ``librgd.so`` (once) and declare the signatures; raise if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with __graft_entry__.build() "
                           "(python -m paper_2607_20791_gb300.build)")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _check(rc: int) -> None:
    if rc != RGD_OK:
        raise RgdError(rc, load_library().rgd_last_error_string().decode())


class _HostTensor:
    """Stands in for the pointer of a tensor that is not on the GPU; :func:`_call`
    refuses the call once every other argument has been checked."""

    def __init__(self, name: str):
        self.name = name


def _call(fn, *args):
    """Call a C entry point unless an argument is a host tensor."""
    for a in args:
        if isinstance(a, _HostTensor):
            raise ValueError(f"{a.name} must be a CUDA tensor")
    return fn(*args)


def _ptr(t, name: str, dtype=None, optional: bool = False, numel: Optional[int] = None):
    """Device pointer of a contiguous CUDA tensor (or a raw int pointer, passed
    through unchecked).  ``numel`` is the number of elements the call will
    touch: a smaller tensor is refused here, since the C side sees only the
    pointer.  A host tensor gives a :class:`_HostTensor`, refused by
    :func:`_call`, so that every argument's type and size is checked first."""
    if t is None:
        if optional:
            return None
        raise ValueError(f"{name} is required")
    if isinstance(t, int):
        return t
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch tensor or an int pointer")
    if dtype is not None and t.dtype not in (dtype if isinstance(dtype, tuple) else (dtype,)):
        raise TypeError(f"{name}: dtype {t.dtype} not accepted")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements, the call needs {numel}")
    if not t.is_cuda:
        return _HostTensor(name)
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        try:
            return torch.cuda.current_stream().cuda_stream
        except (RuntimeError, AssertionError):  # no CUDA device: the call is refused or fails in CUDA
            return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def rgd_version() -> str:
    return load_library().rgd_version().decode()


def rgd_set_wait_limit_ns(limit_ns: int) -> None:
    """Limit of the attention kernel's waits for later calls (0: the default, 2 s)."""
    _check(load_library().rgd_set_wait_limit_ns(int(limit_ns)))


def rgd_prefix_decode_attn_workspace_size(shape: AttnShape) -> int:
    n = load_library().rgd_prefix_decode_attn_workspace_size(ctypes.byref(shape))
    if n == 0:
        raise RgdError(RGD_ERR_INVALID_ARG, load_library().rgd_last_error_string().decode())
    return int(n)


def _attn_sizes(shape: AttnShape) -> dict:
    """Elements each attention argument must hold for ``shape``."""
    R = shape.num_groups * shape.rows_per_group
    return {"q": R * shape.num_q_heads * shape.head_dim,
            "kv": shape.num_pages * shape.num_kv_heads * shape.page_size * shape.head_dim,
            "pbt": shape.num_groups * shape.max_prompt_pages, "plen": shape.num_groups,
            "sbt": R * shape.max_suffix_pages, "rows": R, "lse": R * shape.num_q_heads}


def rgd_prefix_decode_attn(shape: AttnShape, q, k_pages, v_pages, prompt_block_table, prompt_len,
                           suffix_block_table, suffix_len, row_active, softmax_scale: float, out, lse,
                           workspace, dev_status=None, stream=None) -> None:
    import torch
    lib = load_library()
    n = _attn_sizes(shape)
    ws_bytes = workspace.numel() * workspace.element_size() if isinstance(workspace, torch.Tensor) else 0
    _check(_call(lib.rgd_prefix_decode_attn,
        ctypes.byref(shape), _ptr(q, "q", torch.bfloat16, numel=n["q"]),
        _ptr(k_pages, "k_pages", torch.bfloat16, numel=n["kv"]), _ptr(v_pages, "v_pages", torch.bfloat16, numel=n["kv"]),
        _ptr(prompt_block_table, "prompt_block_table", torch.int32, numel=n["pbt"]),
        _ptr(prompt_len, "prompt_len", torch.int32, numel=n["plen"]),
        _ptr(suffix_block_table, "suffix_block_table", torch.int32, numel=n["sbt"]),
        _ptr(suffix_len, "suffix_len", torch.int32, numel=n["rows"]),
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=n["rows"]), float(softmax_scale),
        _ptr(out, "out", torch.bfloat16, numel=n["q"]), _ptr(lse, "lse", torch.float32, optional=True, numel=n["lse"]),
        _ptr(workspace, "workspace"), ws_bytes, _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1),
        _stream(stream)))


def rgd_prefix_decode_attn_noalloc(shape: AttnShape, q, k_pages, v_pages, prompt_block_table, prompt_len,
                                   suffix_block_table, suffix_len, row_active, softmax_scale: float, out,
                                   lse, dev_status=None, stream=None) -> None:
    """Same as :func:`rgd_prefix_decode_attn` without a workspace: the library's
    fixed device scratch is used (for callers that cannot allocate device memory)."""
    import torch
    n = _attn_sizes(shape)
    _check(_call(load_library().rgd_prefix_decode_attn_noalloc,
        ctypes.byref(shape), _ptr(q, "q", torch.bfloat16, numel=n["q"]),
        _ptr(k_pages, "k_pages", torch.bfloat16, numel=n["kv"]), _ptr(v_pages, "v_pages", torch.bfloat16, numel=n["kv"]),
        _ptr(prompt_block_table, "prompt_block_table", torch.int32, numel=n["pbt"]),
        _ptr(prompt_len, "prompt_len", torch.int32, numel=n["plen"]),
        _ptr(suffix_block_table, "suffix_block_table", torch.int32, numel=n["sbt"]),
        _ptr(suffix_len, "suffix_len", torch.int32, numel=n["rows"]),
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=n["rows"]), float(softmax_scale),
        _ptr(out, "out", torch.bfloat16, numel=n["q"]), _ptr(lse, "lse", torch.float32, optional=True, numel=n["lse"]),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def rgd_sample_head(logits, is_probe, temperature, min_p, seed, step: int, row_active, token_out,
                    kept_count=None, kept_mask=None, dev_status=None, stream=None) -> None:
    import torch
    if logits.dim() != 2:
        raise ValueError("logits must be [rows, vocab]")
    dtype = {torch.float32: RGD_F32, torch.bfloat16: RGD_BF16}.get(logits.dtype)
    if dtype is None:
        raise TypeError("logits must be float32 or bfloat16")
    rows, vocab = logits.shape
    _check(_call(load_library().rgd_sample_head,
        rows, vocab, dtype, _ptr(logits, "logits"),
        _ptr(is_probe, "is_probe", torch.uint8, optional=True, numel=rows),
        _ptr(temperature, "temperature", torch.float32, numel=rows), _ptr(min_p, "min_p", torch.float32, numel=rows),
        _ptr(seed, "seed", (torch.int64, torch.uint64), numel=rows), int(step) & 0xFFFFFFFFFFFFFFFF,
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=rows),
        _ptr(token_out, "token_out", torch.int32, numel=rows),
        _ptr(kept_count, "kept_count", torch.int32, optional=True, numel=rows),
        _ptr(kept_mask, "kept_mask", torch.uint8, optional=True, numel=rows * vocab),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def _logits_dtype(logits):
    import torch
    if logits.dim() != 2:
        raise ValueError("logits must be [rows, vocab]")
    dtype = {torch.float32: RGD_F32, torch.bfloat16: RGD_BF16}.get(logits.dtype)
    if dtype is None:
        raise TypeError("logits must be float32 or bfloat16")
    return dtype


def rgd_sample_head_gated(logits, is_probe, temperature, min_p, seed, step: int, row_active, token_out,
                          kept_count, trie: "Trie", rows_per_group: int, eos_token: int, max_len: int, state,
                          dev_status=None, stream=None) -> None:
    """The sample head and the hard gate of one step in one kernel (see the C header)."""
    import torch
    dtype = _logits_dtype(logits)
    rows, vocab = logits.shape
    rpg = int(rows_per_group)
    groups = rows // rpg if rpg > 0 else 0
    _check(_call(load_library().rgd_sample_head_gated,
        rows, vocab, dtype, _ptr(logits, "logits"),
        _ptr(is_probe, "is_probe", torch.uint8, optional=True, numel=rows),
        _ptr(temperature, "temperature", torch.float32, numel=rows), _ptr(min_p, "min_p", torch.float32, numel=rows),
        _ptr(seed, "seed", (torch.int64, torch.uint64), numel=rows), int(step) & 0xFFFFFFFFFFFFFFFF,
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=rows),
        _ptr(token_out, "token_out", torch.int32, numel=rows),
        _ptr(kept_count, "kept_count", torch.int32, optional=True, numel=rows),
        trie.handle, rpg, int(eos_token), int(max_len), _state_ptr(state, groups),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def rgd_decode_step(shape: AttnShape, q, k_pages, v_pages, prompt_block_table, prompt_len, suffix_block_table,
                    suffix_len, softmax_scale: float, out, lse, workspace, logits, is_probe, temperature, min_p,
                    seed, step: int, row_active, token_out, kept_count, trie: "Trie", eos_token: int,
                    max_len: int, state, dev_status=None, stream=None) -> None:
    """One whole decode step: attention, then the gated sample head (see the C header)."""
    import torch
    n = _attn_sizes(shape)
    dtype = _logits_dtype(logits)
    rows, vocab = logits.shape
    if rows != n["rows"]:
        raise ValueError(f"logits has {rows} rows, the attention shape {n['rows']}")
    ws_bytes = workspace.numel() * workspace.element_size() if isinstance(workspace, torch.Tensor) else 0
    _check(_call(load_library().rgd_decode_step,
        ctypes.byref(shape), _ptr(q, "q", torch.bfloat16, numel=n["q"]),
        _ptr(k_pages, "k_pages", torch.bfloat16, numel=n["kv"]), _ptr(v_pages, "v_pages", torch.bfloat16, numel=n["kv"]),
        _ptr(prompt_block_table, "prompt_block_table", torch.int32, numel=n["pbt"]),
        _ptr(prompt_len, "prompt_len", torch.int32, numel=n["plen"]),
        _ptr(suffix_block_table, "suffix_block_table", torch.int32, numel=n["sbt"]),
        _ptr(suffix_len, "suffix_len", torch.int32, numel=n["rows"]), float(softmax_scale),
        _ptr(out, "out", torch.bfloat16, numel=n["q"]), _ptr(lse, "lse", torch.float32, optional=True, numel=n["lse"]),
        _ptr(workspace, "workspace"), ws_bytes, vocab, dtype, _ptr(logits, "logits"),
        _ptr(is_probe, "is_probe", torch.uint8, optional=True, numel=rows),
        _ptr(temperature, "temperature", torch.float32, numel=rows), _ptr(min_p, "min_p", torch.float32, numel=rows),
        _ptr(seed, "seed", (torch.int64, torch.uint64), numel=rows), int(step) & 0xFFFFFFFFFFFFFFFF,
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=rows),
        _ptr(token_out, "token_out", torch.int32, numel=rows),
        _ptr(kept_count, "kept_count", torch.int32, optional=True, numel=rows),
        trie.handle, int(eos_token), int(max_len), _state_ptr(state, shape.num_groups),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


class Trie:
    """Owner of an ``rgd_trie`` handle built from host token sequences."""

    def __init__(self, sequences, min_confirm: int = 2):
        import numpy as np
        lib = load_library()
        seqs = [np.asarray(s, dtype=np.int32).reshape(-1) for s in sequences]
        toks = np.concatenate(seqs) if seqs else np.zeros(1, np.int32)
        offs = np.zeros(len(seqs) + 1, dtype=np.int64)
        for i, s in enumerate(seqs):
            offs[i + 1] = offs[i] + s.size
        toks = np.ascontiguousarray(toks)
        h = _P()
        _check(lib.rgd_trie_create(toks.ctypes.data, offs.ctypes.data, len(seqs), int(min_confirm),
                                   ctypes.byref(h)))
        self.handle = h
        self._lib = lib

    def info(self):
        n, e = _I32(), _I32()
        _check(self._lib.rgd_trie_info(self.handle, ctypes.byref(n), ctypes.byref(e)))
        return n.value, e.value

    def close(self):
        if getattr(self, "handle", None):
            self._lib.rgd_trie_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def rgd_trie_create(sequences, min_confirm: int = 2) -> Trie:
    return Trie(sequences, min_confirm)


def _state_ptr(state, groups: int) -> Optional[int]:
    """A gate-state buffer must hold ``groups`` states of GATE_STATE_BYTES each."""
    import torch
    return _ptr(state, "state", torch.uint8, numel=max(int(groups), 0) * GATE_STATE_BYTES)


def rgd_gate_state_init(state, groups: int, stream=None) -> None:
    _check(_call(load_library().rgd_gate_state_init, _state_ptr(state, groups), int(groups), _stream(stream)))


def rgd_probe_gate(trie: Trie, groups: int, rows_per_group: int, probe_tokens, n_tokens: int,
                   token_stride: int, eos_token: int, max_len: int, state, row_active=None,
                   dev_status=None, stream=None) -> None:
    import torch
    G, rpg = int(groups), int(rows_per_group)
    tok_n = (G - 1) * int(token_stride) + int(n_tokens) if G > 0 else 0
    _check(_call(load_library().rgd_probe_gate,
        trie.handle, G, rpg, _ptr(probe_tokens, "probe_tokens", torch.int32, numel=tok_n),
        int(n_tokens), int(token_stride), int(eos_token), int(max_len), _state_ptr(state, G),
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=G * rpg),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def rgd_residual_precheck(h, w, bias: float, theta: float, rows_per_group: int, state, row_active=None,
                          prob_out=None, dev_status=None, stream=None) -> None:
    import torch
    if h.dim() != 2:
        raise ValueError("h must be [groups, d]")
    dtype = {torch.float32: RGD_F32, torch.bfloat16: RGD_BF16}.get(h.dtype)
    if dtype is None:
        raise TypeError("h must be float32 or bfloat16")
    groups, d = h.shape
    rpg = int(rows_per_group)
    _check(_call(load_library().rgd_residual_precheck,
        int(groups), int(d), dtype, _ptr(h, "h"), _ptr(w, "w", torch.float32, numel=d), float(bias), float(theta),
        rpg, _ptr(prob_out, "prob_out", torch.float32, optional=True, numel=groups), _state_ptr(state, groups),
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=groups * rpg),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def rgd_soft_gate(trie: Trie, groups: int, rows_per_group: int, logits, row_stride: int, top_k: int, rho: float,
                  c: int, eos_token: int, max_len: int, state, token_out, row_active=None, mass_out=None,
                  dev_status=None, stream=None) -> None:
    """``logits`` is the step's [rows, vocab] tensor (or any tensor whose rows
    g * row_stride / vocab hold group g's probe logits)."""
    import torch
    dtype = {torch.float32: RGD_F32, torch.bfloat16: RGD_BF16}.get(logits.dtype)
    if dtype is None:
        raise TypeError("logits must be float32 or bfloat16")
    vocab = logits.shape[-1]
    G, rpg = int(groups), int(rows_per_group)
    log_n = (G - 1) * int(row_stride) + int(vocab) if G > 0 else 0
    _check(_call(load_library().rgd_soft_gate,
        trie.handle, G, rpg, int(vocab), dtype, _ptr(logits, "logits", numel=log_n), int(row_stride),
        int(top_k), float(rho), int(c), int(eos_token), int(max_len), _state_ptr(state, G),
        _ptr(row_active, "row_active", torch.uint8, optional=True, numel=G * rpg),
        _ptr(token_out, "token_out", torch.int32, numel=G),
        _ptr(mass_out, "mass_out", torch.float32, optional=True, numel=G),
        _ptr(dev_status, "dev_status", torch.int32, optional=True, numel=1), _stream(stream)))


def new_gate_state(groups: int, device="cuda"):
    """A device buffer holding ``groups`` gate states (uint8 [groups, 20])."""
    import torch
    return torch.empty((groups, GATE_STATE_BYTES), dtype=torch.uint8, device=device)


def decode_gate_state(buf) -> dict:
    """Host view of a gate-state buffer: dict of numpy arrays per field."""
    import numpy as np
    a = buf.cpu().numpy().reshape(-1, GATE_STATE_BYTES)
    i32 = a[:, :16].copy().view(np.int32).reshape(-1, 4)
    return {"node": i32[:, 0], "length": i32[:, 1], "steps": i32[:, 2], "decisive_step": i32[:, 3],
            "decision": a[:, 16].copy(), "confirmed": a[:, 17].copy(), "done": a[:, 18].copy()}
