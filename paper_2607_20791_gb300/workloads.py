"""Seeded synthetic inputs for the refusal-gated decode step.

This module only draws inputs: prompt/suffix KV pages and block tables, query
vectors, next-token logits, sampling parameters, refusal-prefix sets and greedy
probe token streams.  It holds none of the method's arithmetic (no attention,
no softmax, no sampling, no prefix matching), so both the CUDA path and the
CPU oracle can be fed from it without sharing any computation.

The paper evaluates through vLLM on real models and datasets (Sec. 4.1); none
of those are available, so every workload below is a synthetic stand-in with
the shapes of a Llama-3-8B-style decode step (32 q heads / 8 kv heads, head
dim 128, 16-token KV pages, vocab 128256) and of the sampling settings the
paper uses (temperatures 1.0-3.0, Sec. 4.1; truncation via min-p, Sec. 1).

All bf16 tensors are returned as ``uint16`` bit patterns (numpy has no bf16).
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

PAGE_SIZE = 16


# --------------------------------------------------------------------------
# dtype helpers (input encoding only)
# --------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round-to-nearest-even), as uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def _rng(seed: int, *salt: int) -> np.random.Generator:
    return np.random.default_rng([int(seed), *[int(s) for s in salt]])


# --------------------------------------------------------------------------
# attention inputs
# --------------------------------------------------------------------------
@dataclasses.dataclass
class AttnCase:
    """Inputs of one shared-prefix decode-attention call.

    Rows of group g are ``g*rows_per_group .. (g+1)*rows_per_group-1``; the
    first row of every group is the greedy probe, the rest are sample rows.
    """

    name: str
    num_groups: int
    rows_per_group: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    q: np.ndarray                  # uint16 [R, Hq, D]
    k_pages: Optional[np.ndarray]  # uint16 [num_pages, Hkv, PAGE_SIZE, D]
    v_pages: Optional[np.ndarray]  # uint16 [num_pages, Hkv, PAGE_SIZE, D]
    num_pages: int
    prompt_block_table: np.ndarray  # int32 [G, max_prompt_pages]
    prompt_len: np.ndarray          # int32 [G]
    suffix_block_table: np.ndarray  # int32 [R, max_suffix_pages]
    suffix_len: np.ndarray          # int32 [R]
    row_active: np.ndarray          # uint8 [R]
    softmax_scale: float
    page_size: int = PAGE_SIZE

    @property
    def num_rows(self) -> int:
        return self.num_groups * self.rows_per_group


def make_attn_case(name: str, num_groups: int, rows_per_group: int, num_q_heads: int,
                   num_kv_heads: int, head_dim: int, prompt_lens: Sequence[int],
                   suffix_lens: Sequence[int], seed: int,
                   row_active: Optional[np.ndarray] = None, spare_pages: int = 3,
                   with_kv: bool = True, min_table_cols: int = 1, suffix_room: int = 0) -> AttnCase:
    """Draw Q and paged K/V ~ N(0,1) in bf16 with pages shuffled in the pool.

    Pages of all prompts and suffixes are assigned through a seeded random
    permutation of the pool, so consecutive logical pages are scattered the way
    a paged KV cache is after some serving time.  Unused block-table entries
    hold -1.  ``suffix_room`` extra tokens of pages are assigned to every row's
    suffix (filled like the rest), so that a decode loop can grow the suffixes
    by that many tokens without a new page.
    """
    G, rpg = int(num_groups), int(rows_per_group)
    R = G * rpg
    prompt_lens = np.asarray(prompt_lens, dtype=np.int32).reshape(G)
    suffix_lens = np.asarray(suffix_lens, dtype=np.int32).reshape(R)
    ppages = (prompt_lens + PAGE_SIZE - 1) // PAGE_SIZE
    spages = (suffix_lens + int(suffix_room) + PAGE_SIZE - 1) // PAGE_SIZE
    total = int(ppages.sum() + spages.sum())
    num_pages = total + int(spare_pages)
    rng = _rng(seed, 1)
    perm = rng.permutation(num_pages).astype(np.int32)
    max_pp = max(int(min_table_cols), int(ppages.max()) if G else 0)
    max_sp = max(int(min_table_cols), int(spages.max()) if R else 0)
    pbt = np.full((G, max_pp), -1, dtype=np.int32)
    sbt = np.full((R, max_sp), -1, dtype=np.int32)
    cur = 0
    for g in range(G):
        n = int(ppages[g])
        pbt[g, :n] = perm[cur:cur + n]
        cur += n
    for r in range(R):
        n = int(spages[r])
        sbt[r, :n] = perm[cur:cur + n]
        cur += n
    Hq, Hkv, D = int(num_q_heads), int(num_kv_heads), int(head_dim)
    q = f32_to_bf16_bits(_rng(seed, 2).standard_normal((R, Hq, D), dtype=np.float32))
    k = v = None
    if with_kv:
        shape = (num_pages, Hkv, PAGE_SIZE, D)
        k = _normal_bf16(_rng(seed, 3), shape)
        v = _normal_bf16(_rng(seed, 4), shape)
    if row_active is None:
        row_active = np.ones(R, dtype=np.uint8)
    return AttnCase(name=name, num_groups=G, rows_per_group=rpg, num_q_heads=Hq,
                    num_kv_heads=Hkv, head_dim=D, q=q, k_pages=k, v_pages=v,
                    num_pages=num_pages, prompt_block_table=pbt, prompt_len=prompt_lens,
                    suffix_block_table=sbt, suffix_len=suffix_lens,
                    row_active=np.asarray(row_active, dtype=np.uint8).reshape(R),
                    softmax_scale=1.0 / float(np.sqrt(D)))


def _normal_bf16(rng: np.random.Generator, shape) -> np.ndarray:
    out = np.empty(shape, dtype=np.uint16)
    flat = out.reshape(-1)
    step = 1 << 24
    for i in range(0, flat.size, step):
        n = min(step, flat.size - i)
        flat[i:i + n] = f32_to_bf16_bits(rng.standard_normal(n, dtype=np.float32))
    return out


# --------------------------------------------------------------------------
# sample-head inputs
# --------------------------------------------------------------------------
@dataclasses.dataclass
class HeadCase:
    """Inputs of one sample-head call over ``rows`` rows of next-token logits."""

    name: str
    logits: np.ndarray        # float32 [rows, V] or uint16 bf16 bits [rows, V]
    dtype: str                # "f32" or "bf16"
    is_probe: np.ndarray      # uint8 [rows]
    temperature: np.ndarray   # float32 [rows]
    min_p: np.ndarray         # float32 [rows]
    seed: np.ndarray          # uint64 [rows]
    step: int
    row_active: np.ndarray    # uint8 [rows]

    @property
    def rows(self) -> int:
        return int(self.logits.shape[0])

    @property
    def vocab(self) -> int:
        return int(self.logits.shape[1])


def zipf_logits(rows: int, vocab: int, seed: int, s: float = 1.1,
                noise: float = 1.0) -> np.ndarray:
    """Zipf(s)-ranked log-probabilities plus N(0, noise^2), float32 [rows, vocab].

    Token i of a row gets rank perm[i]+1 from a seeded permutation, and the value
    -s*ln(rank) - ln(H) with H the generalised harmonic number, plus noise.
    """
    ranks = np.arange(1, vocab + 1, dtype=np.float64)
    base = -s * np.log(ranks)
    base -= np.log(np.sum(np.exp(base)))
    out = np.empty((rows, vocab), dtype=np.float32)
    rng = _rng(seed, 5)
    for r in range(rows):
        perm = rng.permutation(vocab)
        out[r] = (base[perm] + noise * rng.standard_normal(vocab)).astype(np.float32)
    return out


def _seeds(rng: np.random.Generator, n: int) -> np.ndarray:
    return rng.integers(0, np.iinfo(np.uint64).max, size=n, dtype=np.uint64, endpoint=True)


def make_head_case(name: str, logits32: np.ndarray, dtype: str, is_probe, temperature,
                   min_p, seed: int, step: int = 0, row_active=None) -> HeadCase:
    rows = logits32.shape[0]
    logits = logits32.astype(np.float32) if dtype == "f32" else f32_to_bf16_bits(logits32)
    if row_active is None:
        row_active = np.ones(rows, dtype=np.uint8)
    return HeadCase(name=name, logits=logits, dtype=dtype,
                    is_probe=np.asarray(is_probe, dtype=np.uint8).reshape(rows),
                    temperature=np.asarray(temperature, dtype=np.float32).reshape(rows),
                    min_p=np.asarray(min_p, dtype=np.float32).reshape(rows),
                    seed=_seeds(_rng(seed, 6), rows), step=int(step),
                    row_active=np.asarray(row_active, dtype=np.uint8).reshape(rows))


# --------------------------------------------------------------------------
# refusal-prefix sets and greedy probe streams
# --------------------------------------------------------------------------
@dataclasses.dataclass
class GateCase:
    """Refusal-prefix set P (token sequences) and per-group greedy probe tokens."""

    name: str
    refusal_seqs: List[np.ndarray]   # each int32 [len]
    tokens: np.ndarray               # int32 [groups, n_steps]
    eos: int                         # -1 = no stop token
    max_len: int                     # L
    rows_per_group: int
    min_confirm: int = 2

    @property
    def groups(self) -> int:
        return int(self.tokens.shape[0])


def make_refusal_set(n: int, min_len: int, max_len: int, vocab: int, seed: int,
                     nested_frac: float = 0.1, dup_frac: float = 0.02,
                     avoid: Sequence[int] = ()) -> List[np.ndarray]:
    """Random token sequences; a fraction are prefixes of others or duplicates."""
    rng = _rng(seed, 7)
    avoid = set(int(a) for a in avoid)
    seqs: List[np.ndarray] = []
    for i in range(n):
        u = rng.random()
        if seqs and u < nested_frac:
            base = seqs[int(rng.integers(len(seqs)))]
            if len(base) > min_len:
                seqs.append(base[:int(rng.integers(min_len, len(base)))].copy())
                continue
        if seqs and u < nested_frac + dup_frac:
            seqs.append(seqs[int(rng.integers(len(seqs)))].copy())
            continue
        L = int(rng.integers(min_len, max_len + 1))
        toks = rng.integers(0, vocab, size=L).astype(np.int32)
        for j in range(L):
            while int(toks[j]) in avoid:
                toks[j] = int(rng.integers(0, vocab))
        seqs.append(toks)
    return seqs


def make_probe_streams(refusal_seqs: Sequence[np.ndarray], groups: int, n_steps: int,
                       vocab: int, seed: int, eos: int = -1) -> np.ndarray:
    """Greedy probe token streams [groups, n_steps] with a planted mix.

    Kinds (cycled over groups): follow a refusal sequence fully then continue at
    random; follow one part-way then diverge; random from the start; follow a
    sequence part-way then emit the stop token (when ``eos >= 0``).
    """
    rng = _rng(seed, 8)
    out = rng.integers(0, vocab, size=(groups, n_steps)).astype(np.int32)
    if eos >= 0:
        out[out == eos] = (eos + 1) % vocab
    for g in range(groups):
        kind = g % 4
        if not refusal_seqs or kind == 2:
            continue
        s = refusal_seqs[int(rng.integers(len(refusal_seqs)))]
        if kind == 0:
            k = min(len(s), n_steps)
        else:
            k = int(rng.integers(0, min(len(s), n_steps)))
        out[g, :k] = s[:k]
        if kind == 3 and eos >= 0 and k < n_steps:
            out[g, k] = eos
    return out


def loop_probe_streams(refusal_seqs: Sequence[np.ndarray], groups: int, n_steps: int, vocab: int,
                       seed: int, eos: int) -> np.ndarray:
    """Greedy probe streams [groups, n_steps] for a whole gated loop, one kind per
    group in turn: (0) a refusal sequence in full, then random tokens to the
    cap; (1) a refusal sequence in full, then random tokens, then the stop token
    at a random later step; (2) part of a sequence, then a diverging token;
    (3) random from the start; (4) a proper prefix of a sequence, then the stop
    token.  Random tokens never equal the stop token."""
    rng = _rng(seed, 9)
    out = rng.integers(0, vocab, size=(groups, n_steps)).astype(np.int32)
    out[out == eos] = (eos + 1) % vocab
    for g in range(groups):
        kind = g % 5
        if kind == 3 or not refusal_seqs:
            continue
        s = refusal_seqs[int(rng.integers(len(refusal_seqs)))]
        if kind in (0, 1):
            k = min(len(s), n_steps)
            out[g, :k] = s[:k]
            if kind == 1 and k + 1 < n_steps:
                out[g, int(rng.integers(k, n_steps))] = eos
        else:
            k = int(rng.integers(1, len(s))) if len(s) > 1 else 0
            k = min(k, n_steps - 1)
            out[g, :k] = s[:k]
            if kind == 4:
                out[g, k] = eos
    return out


# --------------------------------------------------------------------------
# the five workloads
# --------------------------------------------------------------------------
@dataclasses.dataclass
class StepCase:
    """One decode step: attention inputs, sample-head inputs and the gate inputs."""

    name: str
    attn: AttnCase
    head: HeadCase
    gate: GateCase


def _gate_for_step(name, seed, groups, rpg, vocab, n_seq, lmin, lmax, max_len, eos=-1):
    seqs = make_refusal_set(n_seq, lmin, lmax, vocab, seed, avoid=[eos] if eos >= 0 else [])
    toks = make_probe_streams(seqs, groups, 1, vocab, seed, eos=eos)
    return GateCase(name=name, refusal_seqs=seqs, tokens=toks, eos=eos, max_len=max_len,
                    rows_per_group=rpg)


def tiny(seed: int = 0, step: int = 0) -> StepCase:
    """1 prompt of 128 tokens, 1 probe + 2 sample rows, 4 q heads / 1 kv head,
    head dim 64, suffixes 0..16; fp32 logits over 4096 ~ N(0, 3^2) plus one +8
    spike per row; T = 1.5, min-p = 0.1; 8 refusal sequences of length 3-6.

    ``step`` selects the logits and suffix lengths of one of the 16 probe steps;
    the probe row's spike follows a refusal sequence for a seed-dependent number
    of steps so the gate sees confirmations, divergences and random starts.
    """
    G, rpg, V = 1, 3, 4096
    srng = _rng(seed, 20, step)
    attn = make_attn_case("tiny", G, rpg, 4, 1, 64, [128], srng.integers(0, 17, size=G * rpg),
                          seed)
    eos = V - 1
    seqs = make_refusal_set(8, 3, 6, V, seed, avoid=[eos])
    logits = (3.0 * srng.standard_normal((G * rpg, V))).astype(np.float32)
    follow = [len(seqs[0]) + 2, 1, 0][seed % 3]
    spike_tok = srng.integers(0, V - 1, size=G * rpg)
    logits[np.arange(G * rpg), spike_tok] += 8.0
    if step < follow and step < len(seqs[0]):
        # planted probe step: the probe row's spike sits on the next token of a
        # refusal sequence, 8 above the row's maximum so that it is the argmax
        logits[0, int(seqs[0][step])] = logits[0].max() + 8.0
    head = make_head_case("tiny", logits, "f32", [1, 0, 0], [0.0, 1.5, 1.5], [0.1] * 3,
                          seed * 1000 + 17, step=step)
    gate = GateCase(name="tiny", refusal_seqs=seqs, tokens=np.zeros((G, 1), np.int32),
                    eos=eos, max_len=16, rows_per_group=rpg)
    return StepCase("tiny", attn, head, gate)


def llama8b(seed: int = 0, with_kv: bool = True) -> StepCase:
    """Llama-3-8B-shaped step: 16 prompts of U[512, 2048] tokens, 1 probe + 4
    sample rows each, suffixes U[0, 256], 32 q / 8 kv heads, head dim 128, bf16
    KV in 16-token pages; fp32 Zipf(1.1) logits over 128256; temperatures
    {1.0, 1.5, 2.0, 3.0} over the sample rows, min-p {0.05, 0.1} by group; 64
    refusal sequences of length 2-8."""
    G, rpg, V = 16, 5, 128256
    rng = _rng(seed, 21)
    plens = rng.integers(512, 2049, size=G)
    slens = rng.integers(0, 257, size=G * rpg)
    attn = make_attn_case("llama8b", G, rpg, 32, 8, 128, plens, slens, seed, with_kv=with_kv)
    logits = zipf_logits(G * rpg, V, seed)
    is_probe = np.tile([1, 0, 0, 0, 0], G)
    temps = np.tile([0.0, 1.0, 1.5, 2.0, 3.0], G)
    minp = np.repeat([0.05 if g % 2 == 0 else 0.1 for g in range(G)], rpg)
    head = make_head_case("llama8b", logits, "f32", is_probe, temps, minp, seed)
    gate = _gate_for_step("llama8b", seed, G, rpg, V, 64, 2, 8, 128)
    return StepCase("llama8b", attn, head, gate)


def long_prompt(seed: int = 0, with_kv: bool = True) -> StepCase:
    """4 prompts of 32768 tokens, 1 probe + 8 sample rows each, suffixes up to
    1024, 64 q / 8 kv heads, head dim 128, bf16 KV; bf16 Zipf logits over 128256;
    T = 2.0, min-p = 0.05."""
    G, rpg, V = 4, 9, 128256
    rng = _rng(seed, 22)
    slens = rng.integers(0, 1025, size=G * rpg)
    attn = make_attn_case("long_prompt", G, rpg, 64, 8, 128, [32768] * G, slens, seed,
                          with_kv=with_kv)
    logits = zipf_logits(G * rpg, V, seed)
    is_probe = np.tile([1] + [0] * (rpg - 1), G)
    temps = np.where(is_probe == 1, 0.0, 2.0)
    head = make_head_case("long_prompt", logits, "bf16", is_probe, temps, [0.05] * (G * rpg), seed)
    gate = _gate_for_step("long_prompt", seed, G, rpg, V, 64, 2, 8, 128)
    return StepCase("long_prompt", attn, head, gate)


def high_batch(seed: int = 0, with_kv: bool = True, lognormal_sigma: float = 1.0) -> StepCase:
    """256 prompts, lengths log-normal (median 1024, sigma 1.0 in log space, clipped
    to 128-8192), 1 probe + 1 sample row each, 30% of groups with their sample row
    masked (gated off after the probe), suffixes U[0, 256], 32 q / 8 kv heads, head
    dim 128, bf16 KV; bf16 Zipf logits over 152064, T ~ U[0.7, 5.0], min-p ~ U[0, 0.2]."""
    G, rpg, V = 256, 2, 152064
    rng = _rng(seed, 23)
    plens = np.clip(np.round(1024.0 * np.exp(lognormal_sigma * rng.standard_normal(G))),
                    128, 8192).astype(np.int32)
    slens = rng.integers(0, 257, size=G * rpg)
    active = np.ones(G * rpg, dtype=np.uint8)
    gated = rng.permutation(G)[: int(round(0.3 * G))]
    active[gated * rpg + 1] = 0
    attn = make_attn_case("high_batch", G, rpg, 32, 8, 128, plens, slens, seed,
                          row_active=active, with_kv=with_kv)
    logits = zipf_logits(G * rpg, V, seed)
    is_probe = np.tile([1, 0], G)
    temps = np.where(is_probe == 1, 0.0, rng.uniform(0.7, 5.0, size=G * rpg))
    minp = rng.uniform(0.0, 0.2, size=G * rpg)
    head = make_head_case("high_batch", logits, "bf16", is_probe, temps, minp, seed,
                          row_active=active)
    gate = _gate_for_step("high_batch", seed, G, rpg, V, 64, 2, 8, 128)
    return StepCase("high_batch", attn, head, gate)


@dataclasses.dataclass
class LoopCase:
    """A whole gated decode loop (Alg. 1 with the probe and the sample rows of
    each prompt decoding side by side): every row starts at the end of its
    prompt (empty suffix) and appends one token per step it is active, in the
    suffix pages reserved for it; each step's logits are ``head.logits`` with
    the probe row of group g raised to ``spike`` at ``probe_streams[g, step]``,
    so that the greedy probe follows a planted stream."""

    name: str
    attn: AttnCase
    head: HeadCase
    refusal_seqs: List[np.ndarray]
    probe_streams: np.ndarray   # int32 [G, n_steps]
    eos: int
    max_len: int                # L, the probe's length cap
    gate_cap: int               # c of Alg. 1 (does not change the hard gate's outcome)
    n_steps: int
    spike: float = 64.0


def llama8b_loop(seed: int = 0, n_steps: int = 128, with_kv: bool = True) -> LoopCase:
    """The Llama-3-8B-shaped step as a loop of ``n_steps`` decode steps from the
    prompt end: 16 prompts of U[512, 2048] tokens, 1 probe + 4 sample rows each,
    32 q / 8 kv heads, head dim 128; fp32 Zipf logits over 128256 with the
    config's temperatures and min-p; 64 refusal sequences of length 2-8; the
    probe cap L = 128 and the gate cap c = 3 (App. D); the stop token is the
    last vocabulary entry; the probes follow :func:`loop_probe_streams`."""
    G, rpg, V = 16, 5, 128256
    eos = V - 1
    rng = _rng(seed, 24)
    plens = rng.integers(512, 2049, size=G)
    attn = make_attn_case("llama8b_loop", G, rpg, 32, 8, 128, plens, np.zeros(G * rpg, np.int32), seed,
                          with_kv=with_kv, suffix_room=n_steps)
    logits = zipf_logits(G * rpg, V, seed)
    is_probe = np.tile([1, 0, 0, 0, 0], G)
    temps = np.tile([0.0, 1.0, 1.5, 2.0, 3.0], G)
    minp = np.repeat([0.05 if g % 2 == 0 else 0.1 for g in range(G)], rpg)
    head = make_head_case("llama8b_loop", logits, "f32", is_probe, temps, minp, seed)
    seqs = make_refusal_set(64, 2, 8, V, seed, avoid=[eos])
    streams = loop_probe_streams(seqs, G, n_steps, V, seed, eos)
    return LoopCase(name="llama8b_loop", attn=attn, head=head, refusal_seqs=seqs, probe_streams=streams,
                    eos=eos, max_len=128, gate_cap=3, n_steps=n_steps)


def loop_spikes(case: LoopCase):
    """Flat logit indices [n_steps, G] of each step's planted probe tokens and
    the base values they hold outside that step (float32 [n_steps, G])."""
    G, rpg, V = case.attn.num_groups, case.attn.rows_per_group, case.head.vocab
    rows = np.arange(G, dtype=np.int64) * rpg
    idx = rows[None, :] * V + case.probe_streams.T.astype(np.int64)
    base = case.head.logits.reshape(-1)[idx].astype(np.float32)
    return idx, base


def loop_step_logits(case: LoopCase, step: int) -> np.ndarray:
    """The logits of one loop step (a copy of the base with the step's spikes)."""
    out = case.head.logits.copy()
    rpg = case.attn.rows_per_group
    out[np.arange(case.attn.num_groups) * rpg, case.probe_streams[:, step]] = case.spike
    return out


SWEEP_BATCHES = (1, 8, 64, 256, 1024)
SWEEP_VOCABS = (32000, 128256, 262144)
SWEEP_TEMPS = (0.0, 1.0, 2.0, 5.0, 10.0)
SWEEP_MINP = (0.0, 0.05, 0.1, 0.3)


def head_sweep(batch: int, vocab: int, dtype: str, seed: int = 0) -> HeadCase:
    """Logits-only rows: Zipf-ranked logits with N(0,1) noise; temperatures cycle
    over {0 (greedy), 1, 2, 5, 10} and min-p over {0, 0.05, 0.1, 0.3}."""
    logits = zipf_logits(batch, vocab, seed)
    t = np.array([SWEEP_TEMPS[i % len(SWEEP_TEMPS)] for i in range(batch)], np.float32)
    m = np.array([SWEEP_MINP[(i // len(SWEEP_TEMPS)) % len(SWEEP_MINP)] for i in range(batch)],
                 np.float32)
    return make_head_case(f"sweep_b{batch}_v{vocab}_{dtype}", logits, dtype,
                          np.zeros(batch, np.uint8), t, m, seed)


def gate_sweep(groups: int = 1024, n_seq: int = 1000, vocab: int = 128256, n_steps: int = 32,
               seed: int = 0, eos: int = -1) -> GateCase:
    """Refusal trie of ``n_seq`` random sequences of length 2-12 matched against
    ``n_steps``-token greedy probes with a planted mix of behaviours."""
    seqs = make_refusal_set(n_seq, 2, 12, vocab, seed, avoid=[eos] if eos >= 0 else [])
    toks = make_probe_streams(seqs, groups, n_steps, vocab, seed, eos=eos)
    return GateCase(name=f"gate_g{groups}_n{n_seq}", refusal_seqs=seqs, tokens=toks, eos=eos,
                    max_len=n_steps, rows_per_group=1)


@dataclasses.dataclass
class PrecheckCase:
    """Inputs of the residual-stream precheck (App. A): one last-prompt-token
    activation per group, a logistic readout (w, b) and the skip threshold."""
    name: str
    h: np.ndarray        # float32 [G, d] or uint16 bf16 bits [G, d]
    dtype: str           # "f32" or "bf16"
    w: np.ndarray        # float32 [d]
    b: float
    theta: float
    rows_per_group: int

    @property
    def groups(self) -> int:
        return self.h.shape[0]

    @property
    def d(self) -> int:
        return self.h.shape[1]


def make_precheck_case(name: str, groups: int, d: int, dtype: str, theta: float, seed: int,
                       weight_scale: float = 1.0, bias: float = 0.0, rows_per_group: int = 5) -> PrecheckCase:
    """Activations ~ N(0, 1) (fp32, or rounded to bf16), weights ~ N(0, weight_scale^2 / d)
    in fp32, so that the readout's spread across groups is about weight_scale."""
    h32 = _rng(seed, 41).standard_normal((groups, d), dtype=np.float32)
    h = h32 if dtype == "f32" else f32_to_bf16_bits(h32)
    w = (_rng(seed, 42).standard_normal(d) * (weight_scale / np.sqrt(d))).astype(np.float32)
    return PrecheckCase(name=name, h=h, dtype=dtype, w=w, b=float(bias), theta=float(theta),
                        rows_per_group=rows_per_group)


def llama8b_precheck(seed: int = 0) -> PrecheckCase:
    """The Llama-3-8B-shaped step's 16 prompt groups: d = 4096 bf16 activations,
    the paper's calibrated Llama threshold theta = 1e-5, a readout spread of 8 so
    that a few groups fall under it."""
    return make_precheck_case("llama8b_precheck", 16, 4096, "bf16", 1e-5, seed, weight_scale=8.0,
                              bias=-2.0, rows_per_group=5)


CONFIGS = {
    "tiny": tiny,
    "llama8b": llama8b,
    "long_prompt": long_prompt,
    "high_batch": high_batch,
}
