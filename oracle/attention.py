"""Decode attention over shared prompt KV + per-row suffix KV, oracle side (test infrastructure only).

What the shared-prefix path computes (Sec. 3: the prompt KV cache is computed once
and reused by the greedy probe and by high-temperature sampling): every row r of
prompt group g attends, for each query head j, over the concatenation of

* the P_g tokens of the group's prompt KV (shared by all rows of the group), and
* the S_r tokens of the row's own generated suffix KV,

o[r, j] = softmax(scale * K q[r, j]) V with K, V the concatenated keys / values of
kv head h = j // (Hq / Hkv) (consecutive query heads share a kv head -- the usual
grouped-query mapping; the paper is silent), scale = 1/sqrt(D) unless given, and
lse[r, j] = ln(sum exp(scale * K q[r, j])).  No causal mask: a decode query sees
every listed token.  No rotary embedding is applied (inputs are already
positioned).  P_g = S_r = 0 gives o = 0 and lse = -inf.

Token t of a sequence lives in page table[t // page_size], slot t % page_size of
the paged pools k_pages / v_pages [num_pages, Hkv, page_size, D].

This is the plain definition (fp64 from the bf16 inputs); the split-KV / log-sum-
exp-merged kernel reaches the same result up to rounding.  Pinned by closed forms
(single token, equal keys, a two-token hand example), page-shuffle invariance,
torch's CPU scaled_dot_product_attention in fp64, and the log-sum-exp split
identity (tests/test_oracle_attention.py).
"""
from __future__ import annotations

import numpy as np

from .sampling import bf16_bits_to_f32


def gather_tokens(pages: np.ndarray, table_row: np.ndarray, n_tokens: int, kv_head: int,
                  page_size: int) -> np.ndarray:
    """Tokens 0..n_tokens-1 of one sequence for one kv head, as fp64 [n_tokens, D]."""
    D = pages.shape[-1]
    out = np.empty((n_tokens, D), dtype=np.float64)
    for t in range(0, n_tokens, page_size):
        page = int(table_row[t // page_size])
        n = min(page_size, n_tokens - t)
        out[t:t + n] = bf16_bits_to_f32(pages[page, kv_head, :n, :])
    return out


def decode_attention(q, k_pages, v_pages, prompt_block_table, prompt_len, suffix_block_table,
                     suffix_len, rows_per_group: int, num_kv_heads: int, scale=None,
                     page_size: int = 16, rows=None):
    """Return (o fp64 [R, Hq, D], lse fp64 [R, Hq]) for the listed rows (default all)."""
    R, Hq, D = q.shape
    gq = Hq // num_kv_heads
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    o = np.zeros((R, Hq, D), dtype=np.float64)
    lse = np.full((R, Hq), -np.inf, dtype=np.float64)
    qf = bf16_bits_to_f32(q).astype(np.float64)
    for r in (range(R) if rows is None else rows):
        g = r // rows_per_group
        for h in range(num_kv_heads):
            kp = gather_tokens(k_pages, prompt_block_table[g], int(prompt_len[g]), h, page_size)
            vp = gather_tokens(v_pages, prompt_block_table[g], int(prompt_len[g]), h, page_size)
            ks = gather_tokens(k_pages, suffix_block_table[r], int(suffix_len[r]), h, page_size)
            vs = gather_tokens(v_pages, suffix_block_table[r], int(suffix_len[r]), h, page_size)
            K = np.concatenate([kp, ks], axis=0)
            V = np.concatenate([vp, vs], axis=0)
            if K.shape[0] == 0:
                continue
            for j in range(h * gq, (h + 1) * gq):
                s = scale * (K @ qf[r, j])
                m = s.max()
                e = np.exp(s - m)
                o[r, j] = (e @ V) / e.sum()
                lse[r, j] = m + np.log(e.sum())
    return o, lse


def decode_attention_case(case, rows=None):
    """:func:`decode_attention` on a ``workloads.AttnCase``."""
    return decode_attention(case.q, case.k_pages, case.v_pages, case.prompt_block_table,
                            case.prompt_len, case.suffix_block_table, case.suffix_len,
                            case.rows_per_group, case.num_kv_heads, case.softmax_scale,
                            case.page_size, rows=rows)
