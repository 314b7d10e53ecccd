"""Greedy step and truncated high-temperature sampler, oracle side (test infrastructure only).

Follows the paper's decode primitives (Sec. 3, Alg. 1):

* G_M(p, q): one greedy decode step -> the argmax of the next-token logits.
  Ties are broken toward the lowest token index.
* S_{T,theta}(M, p): plain sampling at a high temperature T, truncated as the
  parameters theta say.  The truncation used here is min-p (cited in
  Sec. 1 and Sec. 2): keep the tokens whose probability under softmax(l / T) is
  at least p_min times the largest probability, renormalise, draw one token.

Step order (a reading: the paper runs p-less sampling, Sec. 4.1, and defines
neither sampler; the order "temperature, then min-p, then draw" is taken):

1. T == 0 or probe row: token = argmax (lowest index on ties); no draw.
2. l_max = max_i l_i (logits are fp32 or bf16, both exact in fp32).
3. theta32 = fl32(T * ln(p_min)) computed in fp64 and rounded once to fp32
   (p_min = 0 gives -inf); cutoff c = fl32(l_max + theta32); kept set
   K = {i : l_i >= c}, compared in fp32.  Because p_i / p_max =
   exp((l_i - l_max) / T), this is the set {p_i >= p_min * p_max} up to the
   rounding of the cutoff; :func:`kept_set_exact` gives the fp64 set and
   :func:`kept_set_margin` the distance of each token from the exact threshold.
4. w_i = exp((l_i - l_max) / T) for i in K (fp64), Z = sum of w over K,
   C_k = sum of w_j over j in K, j <= k (ascending index).
5. u = Philox uniform for (seed, step); token = smallest k in K with C_k > u*Z.
6. A row is a boundary case when u*Z lies within 1e-6*Z of C_tok or of the
   cumulative sum just before tok; the draw there is decided by rounding and a
   mismatch against another implementation is allowed (and counted).
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .philox import uniform24

BOUNDARY_REL = 1e-6


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns (uint16) to float32 exactly."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32)


def logits_as_f32(logits: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "f32":
        return np.asarray(logits, dtype=np.float32)
    if dtype == "bf16":
        return bf16_bits_to_f32(logits)
    raise ValueError(dtype)


def greedy_token(row: np.ndarray) -> int:
    """G_M: argmax with lowest-index tie-break (np.argmax returns the first maximum)."""
    return int(np.argmax(np.asarray(row, dtype=np.float64)))


def cutoff32(l_max32: np.float32, temperature: float, min_p: float) -> np.float32:
    """c = fl32(l_max + fl32(T * ln p_min)); -inf when p_min == 0."""
    t = float(np.float32(temperature))
    m = float(np.float32(min_p))
    if m <= 0.0:
        return np.float32(-np.inf)
    theta32 = np.float32(t * np.log(m))
    with np.errstate(over="ignore"):
        return np.float32(np.float32(l_max32) + theta32)


def kept_set(row32: np.ndarray, temperature: float, min_p: float) -> np.ndarray:
    """Boolean mask of the min-p kept set in the fp32 statement of step 3."""
    row32 = np.asarray(row32, dtype=np.float32)
    c = cutoff32(row32.max(), temperature, min_p)
    return row32 >= c


def kept_set_exact(row32: np.ndarray, temperature: float, min_p: float) -> np.ndarray:
    """The paper-level set {p_i >= p_min * p_max} with p = softmax(l / T), in fp64."""
    l = np.asarray(row32, dtype=np.float64)
    t = float(np.float32(temperature))
    m = float(np.float32(min_p))
    z = (l - l.max()) / t
    p = np.exp(z) / np.sum(np.exp(z))
    return p >= m * p.max()


def kept_set_margin(row32: np.ndarray, temperature: float, min_p: float) -> np.ndarray:
    """Per token: (l_i - l_max)/T - ln p_min in fp64 (>= 0 means kept exactly)."""
    l = np.asarray(row32, dtype=np.float64)
    t = float(np.float32(temperature))
    m = float(np.float32(min_p))
    if m <= 0.0:
        return np.full(l.shape, np.inf)
    return (l - l.max()) / t - np.log(m)


@dataclasses.dataclass
class SampleResult:
    token: int
    kept: np.ndarray       # bool mask over the vocabulary (None for greedy rows)
    kept_count: int
    boundary: bool         # u*Z within BOUNDARY_REL*Z of a CDF step next to the token
    u: float


def sample_from_uniform(row32: np.ndarray, temperature: float, min_p: float,
                        u: float) -> SampleResult:
    """Steps 2-6 for one row, given the uniform u in [0, 1)."""
    row32 = np.asarray(row32, dtype=np.float32)
    kept = kept_set(row32, temperature, min_p)
    idx = np.nonzero(kept)[0]
    l = row32.astype(np.float64)
    t = float(np.float32(temperature))
    w = np.exp((l[idx] - l.max()) / t)
    cdf = np.cumsum(w)
    Z = float(cdf[-1])
    target = u * Z
    k = int(np.searchsorted(cdf, target, side="right"))  # first C_k > target
    k = min(k, idx.size - 1)
    tok = int(idx[k])
    before = float(cdf[k - 1]) if k > 0 else 0.0
    boundary = (abs(target - float(cdf[k])) <= BOUNDARY_REL * Z
                or abs(target - before) <= BOUNDARY_REL * Z)
    return SampleResult(token=tok, kept=kept, kept_count=int(idx.size), boundary=boundary, u=u)


def sample_row(row32: np.ndarray, is_probe: bool, temperature: float, min_p: float,
               seed: int, step: int) -> SampleResult:
    """One row of the sample head: greedy for probe rows and T == 0, else steps 2-6."""
    row32 = np.asarray(row32, dtype=np.float32)
    if is_probe or float(temperature) == 0.0:
        return SampleResult(token=greedy_token(row32), kept=None, kept_count=1,
                            boundary=False, u=float("nan"))
    return sample_from_uniform(row32, temperature, min_p, uniform24(seed, step))


@dataclasses.dataclass
class HeadResult:
    tokens: np.ndarray       # int32 [rows]; -1 for inactive rows
    kept_count: np.ndarray   # int32 [rows]; 0 for inactive rows
    boundary: np.ndarray     # bool [rows]
    kept: list               # per row: bool mask or None


def sample_head(logits: np.ndarray, dtype: str, is_probe, temperature, min_p, seed, step: int,
                row_active=None, rows=None) -> HeadResult:
    """The sample head over all (or the listed) rows."""
    l32 = logits_as_f32(logits, dtype)
    n = l32.shape[0]
    active = np.ones(n, np.uint8) if row_active is None else np.asarray(row_active)
    tokens = np.full(n, -1, np.int32)
    counts = np.zeros(n, np.int32)
    boundary = np.zeros(n, bool)
    kept = [None] * n
    for r in (range(n) if rows is None else rows):
        if not active[r]:
            continue
        res = sample_row(l32[r], bool(is_probe[r]), float(temperature[r]), float(min_p[r]),
                         int(seed[r]), step)
        tokens[r] = res.token
        counts[r] = res.kept_count
        boundary[r] = res.boundary
        kept[r] = res.kept
    return HeadResult(tokens=tokens, kept_count=counts, boundary=boundary, kept=kept)
