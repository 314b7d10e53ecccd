"""Device-side buffers for the seeded workloads (allocation and copies only).

Moves a :class:`workloads.AttnCase` / :class:`workloads.HeadCase` to the GPU as
torch tensors laid out the way the C ABI expects, and allocates the outputs and
the attention workspace.  No arithmetic of the method happens here.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

from . import binding
from .workloads import AttnCase, HeadCase, loop_spikes


def _t(a: np.ndarray, device, dtype=None):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.view(dtype)
    return t.to(device)


@dataclasses.dataclass
class DeviceAttn:
    shape: binding.AttnShape
    q: object
    k_pages: object
    v_pages: object
    prompt_block_table: object
    prompt_len: object
    suffix_block_table: object
    suffix_len: object
    row_active: object
    softmax_scale: float
    out: object
    lse: object
    workspace: object
    dev_status: object

    def run(self, stream=None):
        binding.rgd_prefix_decode_attn(self.shape, self.q, self.k_pages, self.v_pages,
                                       self.prompt_block_table, self.prompt_len,
                                       self.suffix_block_table, self.suffix_len, self.row_active,
                                       self.softmax_scale, self.out, self.lse, self.workspace,
                                       self.dev_status, stream)


def attn_shape(case: AttnCase, num_ctas: int = 0) -> binding.AttnShape:
    return binding.AttnShape(
        num_groups=case.num_groups, rows_per_group=case.rows_per_group,
        num_q_heads=case.num_q_heads, num_kv_heads=case.num_kv_heads, head_dim=case.head_dim,
        page_size=case.page_size, num_pages=case.num_pages,
        max_prompt_pages=case.prompt_block_table.shape[1],
        max_suffix_pages=case.suffix_block_table.shape[1],
        num_ctas=num_ctas, reserved=0)


def attn_to_device(case: AttnCase, device="cuda", num_ctas: int = 0,
                   kv: Optional[tuple] = None) -> DeviceAttn:
    """Copy the case to `device`; `kv` may supply already-resident (k_pages, v_pages)."""
    import torch
    shape = attn_shape(case, num_ctas)
    if kv is None:
        k = _t(case.k_pages, device, torch.bfloat16)
        v = _t(case.v_pages, device, torch.bfloat16)
    else:
        k, v = kv
    R, Hq, D = case.num_rows, case.num_q_heads, case.head_dim
    ws_bytes = binding.rgd_prefix_decode_attn_workspace_size(shape)
    return DeviceAttn(
        shape=shape, q=_t(case.q, device, torch.bfloat16), k_pages=k, v_pages=v,
        prompt_block_table=_t(case.prompt_block_table, device), prompt_len=_t(case.prompt_len, device),
        suffix_block_table=_t(case.suffix_block_table, device), suffix_len=_t(case.suffix_len, device),
        row_active=_t(case.row_active, device), softmax_scale=case.softmax_scale,
        out=torch.zeros((R, Hq, D), dtype=torch.bfloat16, device=device),
        lse=torch.full((R, Hq), float("nan"), dtype=torch.float32, device=device),
        workspace=torch.zeros(ws_bytes, dtype=torch.uint8, device=device),
        dev_status=torch.zeros(1, dtype=torch.int32, device=device))


@dataclasses.dataclass
class DeviceHead:
    logits: object
    is_probe: object
    temperature: object
    min_p: object
    seed: object
    step: int
    row_active: object
    token_out: object
    kept_count: object
    kept_mask: object
    dev_status: object

    def run(self, stream=None, with_mask: bool = True):
        binding.rgd_sample_head(self.logits, self.is_probe, self.temperature, self.min_p, self.seed,
                                self.step, self.row_active, self.token_out, self.kept_count,
                                self.kept_mask if with_mask else None, self.dev_status, stream)


def head_to_device(case: HeadCase, device="cuda", with_mask: bool = False) -> DeviceHead:
    import torch
    rows, V = case.rows, case.vocab
    logits = (_t(case.logits, device) if case.dtype == "f32"
              else _t(case.logits, device, torch.bfloat16))
    return DeviceHead(
        logits=logits, is_probe=_t(case.is_probe, device), temperature=_t(case.temperature, device),
        min_p=_t(case.min_p, device), seed=_t(case.seed.view(np.int64), device), step=case.step,
        row_active=_t(case.row_active, device),
        token_out=torch.full((rows,), -7, dtype=torch.int32, device=device),
        kept_count=torch.full((rows,), -7, dtype=torch.int32, device=device),
        kept_mask=(torch.zeros((rows, V), dtype=torch.uint8, device=device) if with_mask else None),
        dev_status=torch.zeros(1, dtype=torch.int32, device=device))


class DeviceLoop:
    """Device buffers and the captured CUDA graph of a whole gated loop
    (:class:`workloads.LoopCase`): per step, the step's probe tokens are planted
    in the logits, one rgd_decode_step runs (its tokens kept per step, its
    attention output too when ``keep_history``), the logits go back to the
    base, and every row active in the step grows its suffix by one token (the
    KV of that token is already in the row's reserved pages).  A replay starts
    from the prompt end: fresh gate states, every row active, empty suffixes."""

    def __init__(self, case, stream, keep_history=True, kv=None):
        import torch
        self.case = case
        a, h = case.attn, case.head
        G, rpg, n = a.num_groups, a.rows_per_group, case.n_steps
        R = G * rpg
        self.att = attn_to_device(a, kv=kv)
        self.head = head_to_device(h)
        self.trie = binding.Trie(case.refusal_seqs, 2)
        self.state = binding.new_gate_state(G)
        self.row_active = torch.ones(R, dtype=torch.uint8, device="cuda")
        self.snap = torch.empty_like(self.row_active)
        self.suffix_len = torch.zeros(R, dtype=torch.int32, device="cuda")
        idx, base = loop_spikes(case)
        self.idx = torch.from_numpy(idx).cuda()
        self.base = torch.from_numpy(base).cuda()
        self.spike = torch.full((G,), case.spike, dtype=torch.float32, device="cuda")
        self.flat = self.head.logits.view(-1)
        self.tok = torch.full((n, R), -7, dtype=torch.int32, device="cuda")
        self.out = (torch.zeros((n, R, a.num_q_heads, a.head_dim), dtype=torch.bfloat16, device="cuda")
                    if keep_history else None)
        self.status = torch.zeros(1, dtype=torch.int32, device="cuda")
        self.stream = stream
        self.graph = None

    def _body(self):
        s = self.stream.cuda_stream
        a, c = self.att, self.case
        binding.rgd_gate_state_init(self.state, a.shape.num_groups, stream=s)
        self.row_active.fill_(1)
        self.suffix_len.zero_()
        for t in range(c.n_steps):
            self.snap.copy_(self.row_active)
            self.flat.scatter_(0, self.idx[t], self.spike)  # this step's probe tokens
            out = self.out[t] if self.out is not None else a.out
            binding.rgd_decode_step(a.shape, a.q, a.k_pages, a.v_pages, a.prompt_block_table, a.prompt_len,
                                    a.suffix_block_table, self.suffix_len, a.softmax_scale, out, None,
                                    a.workspace, self.head.logits, self.head.is_probe, self.head.temperature,
                                    self.head.min_p, self.head.seed, t, self.row_active, self.tok[t], None,
                                    self.trie, c.eos, c.max_len, self.state, self.status, stream=s)
            self.flat.scatter_(0, self.idx[t], self.base[t])  # back to the base logits
            self.suffix_len.add_(self.snap)  # every row active this step appended its token

    def capture(self):
        import torch
        with torch.cuda.stream(self.stream):
            self._body()  # eager run first (kernel attributes are set outside capture)
            torch.cuda.synchronize()
            self.graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(self.graph, stream=self.stream):
                self._body()
        torch.cuda.synchronize()

    def close(self):
        self.trie.close()
