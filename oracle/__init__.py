"""CPU oracle for the refusal-gated decode step -- TEST INFRASTRUCTURE ONLY.

A plain, slow, obviously correct fp64 NumPy restatement of what the decode-step
hot path computes, written from the paper (arxiv 2607.20791, "Refusal-Gated
Decoding") and the published definitions it relies on:

* ``attention``  -- decode attention of every row over the concatenation of its
  group's shared prompt KV and its own generated-suffix KV (Sec. 3: the prompt KV
  cache is reused across the greedy probe and high-temperature sampling).
* ``sampling``   -- the greedy step G_M (argmax, lowest index on ties) and the
  high-temperature truncated sampler S_{T,theta} as temperature + min-p + an
  inverse-CDF draw (Sec. 3, Alg. 1; min-p cited in Sec. 1 / Sec. 2).
* ``philox``     -- Philox4x32-10 (Salmon et al., SC'11), the counter-based
  generator that supplies the sampler's uniform draw.
* ``gate``       -- the compatibility predicate C(d(q), P) (Sec. 3) on token
  sequences with the two-token minimum for token-prefix detections (App. D),
  as a naive scan over the refusal list, and the per-token hard-gate outcome of
  Alg. 1.
* ``soft_gate``  -- one probe step of the soft compatibility gate of the
  appendix ablation (Alg. 2): top-K, the compatible mass m against rho, a*.
* ``precheck``   -- the residual-stream classifier of App. A: a d + 1 logistic
  readout per prompt and the skip rule p <= theta, applied to the gate state.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline /
reference legs may import this package.  The product library never calls it and
shares no code with it; the two meet only through the seeded input generators.

Parity status of each function is stated in its docstring; every function here
is pinned by ``tests/test_oracle_*.py`` against closed forms, library routines,
published known-answer vectors, brute force or the paper's worked examples,
and ``tests/test_oracle_mutants.py`` checks that those pins catch plausible
mistakes planted in copies of these modules.
"""
