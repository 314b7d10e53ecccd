"""GB300-native decode step of refusal-gated decoding (arxiv 2607.20791).

The compute lives in ``librgd.so`` (CUDA kernels for sm_103a behind the C ABI
in ``include/rgd.h``); :mod:`.binding` is a thin ctypes layer with the same
function names; :mod:`.device` moves the seeded synthetic workloads of
:mod:`.workloads` to the GPU.  Importing the package does not load the library;
the first call does, and raises if it has not been built.
"""
from .binding import (  # noqa: F401
    AttnShape, GateState, RgdError, Trie, decode_gate_state, load_library, new_gate_state,
    rgd_gate_state_init, rgd_prefix_decode_attn, rgd_prefix_decode_attn_workspace_size,
    rgd_probe_gate, rgd_sample_head, rgd_trie_create, rgd_version,
    RGD_PENDING, RGD_REFUSAL, RGD_NON_REFUSAL, RGD_F32, RGD_BF16,
    RGD_DEV_BAD_PAGE, RGD_DEV_BAD_TOKEN, RGD_DEV_WAIT_TIMEOUT, RGD_DEV_BAD_PARAM,
)
