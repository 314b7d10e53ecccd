"""Soft compatibility gate (the appendix ablation's Alg. 2), oracle side (test
infrastructure only).

In the first c probe steps the soft gate relaxes the hard rule of Alg. 1:
when appending the greedy token y leaves the refusal-prefix set, it looks at
the top-K next-token probabilities A; if the refusal-compatible ones (A_ref)
carry probability mass m >= rho, it appends the most probable of them, a*,
and the probe goes on; otherwise the probe is discarded (the prompt is
sampled).  After the first c steps the hard gate applies unchanged.

Readings (the algorithm states these only implicitly):
* P(a) is the model's next-token distribution, softmax of the raw logits
  (temperature 1: the probe is the greedy G_M step whose top-K it reads);
* top-K orders tokens by logit, larger first, the lower index first among
  equal logits (the greedy argmax's own tie rule);
* a* is the first of A_ref in that order (the highest probability, ties to
  the lower index);
* the stop token is handled as by the hard gate: d(q) drops it, so q || eos
  is compatible whenever q is (as the greedy token, and as a top-K
  candidate), and appending it ends the probe;
* the probe goes on with a* (the caller feeds a* back as the probe's token).

Everything is fp64.  States are oracle.gate.GateState; the per-step outcome
of the soft branch is reported for parity (m, A_ref, a*).  Pinned in
tests/test_oracle_soft_gate.py against the appendix's worked illustration on
a toy vocabulary (tests/golden/soft_gate_example.txt), the limits K = 1 and
rho > 1 (the hard gate), and brute force over all compatible candidates.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

from oracle import gate as ogate


@dataclasses.dataclass
class SoftStep:
    token: Optional[int]      # the token appended to the probe (y or a*), None if none
    soft: bool                # the soft branch ran (y incompatible inside the window)
    mass: float = 0.0         # m, the compatible top-K probability mass (soft branch)
    a_ref: List[int] = dataclasses.field(default_factory=list)


def softmax(logits: np.ndarray) -> np.ndarray:
    l = np.asarray(logits, dtype=np.float64)
    e = np.exp(l - l.max())
    return e / e.sum()


def top_k(logits: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k largest logits, larger first, lower index first on ties."""
    l = np.asarray(logits, dtype=np.float64)
    order = np.lexsort((np.arange(l.size), -l))
    return order[:k]


def soft_gate_step(st: ogate.GateState, logits: np.ndarray, P: Sequence[Sequence[int]], eos: int,
                   max_len: int, c: int, k: int, rho: float, min_confirm: int = 2) -> SoftStep:
    """One probe step of the soft gate on the probe's logits (state in place)."""
    if st.done:
        return SoftStep(token=None, soft=False)
    l = np.asarray(logits, dtype=np.float64)
    y = int(np.argmax(l))  # numpy's argmax returns the first (lowest) index of the maximum
    in_window = st.steps < c
    stop = eos >= 0 and y == eos
    if not in_window or stop or ogate.compatible(st.q + [y], P, min_confirm):
        ogate.gate_step(st, y, P, eos, max_len, min_confirm)
        return SoftStep(token=y, soft=False)
    p = softmax(l)
    a_ref = [int(a) for a in top_k(l, k)
             if (eos >= 0 and int(a) == eos) or ogate.compatible(st.q + [int(a)], P, min_confirm)]
    m = float(sum(p[a] for a in a_ref))
    if a_ref and m >= rho:
        a_star = a_ref[0]
        ogate.gate_step(st, a_star, P, eos, max_len, min_confirm)
        return SoftStep(token=a_star, soft=True, mass=m, a_ref=a_ref)
    # no refusal-like alternative with enough mass: discard the probe
    st.decision = ogate.NON_REFUSAL
    st.decisive_step = st.steps
    st.steps += 1
    st.done = True
    return SoftStep(token=None, soft=True, mass=m, a_ref=a_ref)
