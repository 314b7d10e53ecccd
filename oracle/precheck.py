"""Residual-stream precheck, oracle side (test infrastructure only).

App. A replaces the greedy probe of a prompt, when a linear classifier on the
residual stream says a refusal is unlikely: a logistic regression with d + 1
parameters reads the d-dimensional activation h of the prompt's last token at
one layer, and the probe is skipped (the prompt goes straight to
high-temperature sampling) when the predicted refusal probability is at most the calibrated
threshold theta.

    z = w . h + b,   p = sigmoid(z) = 1 / (1 + exp(-z)),   skip  <=>  p <= theta

Everything here is fp64 from the given inputs (h in bf16 is widened exactly).
A skipped group's gate state becomes the outcome of Alg. 1's non-refusal
branch before any probe token: decision NON_REFUSAL, the probe ended, no
decisive token (decisive_step stays -1); its probe row is switched off and its
sample rows go on.  Groups whose state is no longer the fresh empty probe are
left alone (the precheck runs once, before the probe's first token).

Pinned by closed forms and special cases in tests/test_oracle_precheck.py
(w = 0 or h = 0 gives sigmoid(b); the logistic function's symmetry and its
agreement with the library logistic routine; a hand-computed 3-d case;
threshold 0 and 1 extremes).
"""
from __future__ import annotations

from typing import List

import numpy as np

from oracle import gate as ogate


def logits(h: np.ndarray, w: np.ndarray, b: float) -> np.ndarray:
    """z_g = sum_i w_i h_{g,i} + b for every row g of h ([G, d]), fp64."""
    h64 = np.asarray(h, dtype=np.float64)
    w64 = np.asarray(w, dtype=np.float64)
    return h64 @ w64 + float(b)


def sigmoid(z: np.ndarray) -> np.ndarray:
    """1 / (1 + exp(-z)), written per sign so that neither branch overflows."""
    z = np.asarray(z, dtype=np.float64)
    out = np.empty_like(z)
    pos = z >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-z[pos]))
    ez = np.exp(z[~pos])
    out[~pos] = ez / (1.0 + ez)
    return out


def precheck(h: np.ndarray, w: np.ndarray, b: float, theta: float):
    """(z, p, skip) for every group."""
    z = logits(h, w, b)
    p = sigmoid(z)
    return z, p, p <= float(theta)


def apply(states: List[ogate.GateState], skip: np.ndarray, rows_per_group: int,
          row_active: np.ndarray) -> np.ndarray:
    """Gate states and row mask after the precheck (states updated in place)."""
    out = np.array(row_active, dtype=np.uint8, copy=True)
    for g, st in enumerate(states):
        fresh = st.decision == ogate.PENDING and st.steps == 0 and not st.done
        if skip[g] and fresh:
            st.decision = ogate.NON_REFUSAL
            st.done = True
            out[g * rows_per_group] = 0
    return out
