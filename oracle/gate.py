"""Refusal-prefix compatibility gate, oracle side (test infrastructure only).

Compatibility predicate (Sec. 3): C(d(q), P) holds iff d(q) begins some pi in
P, or d(q) itself begins with some pi in P.  It is evaluated here
on token sequences (the runtime detector's token-prefix matching, App. D), with
the two-token minimum of App. D read as: a detection "pi is a prefix of q"
counts only for |pi| >= min_confirm (= 2).  So

    C(q, P) = exists pi in P:  q is a prefix of pi
                            or (pi is a prefix of q and |pi| >= min_confirm).

The probe q is the greedy token sequence after the prompt.  The stop token is
not part of q: d(q) drops special tokens, so appending the stop token does not
change the predicate (a reading; the paper appends y and then tests C(d(q))).

Hard gate, per probe token (Sec. 3 and Alg. 1).  With the hard gate the same
predicate is applied after every probe token, both in the first c gate tokens
and in the post-cap probe B_M, so the cap c does not change the outcome:

* token y is the stop token: the probe ends; the outcome is REFUSAL when
  C(q, P) holds, else NON_REFUSAL (only possible for q = [] and P empty);
* otherwise q <- q || y; if not C(q, P): NON_REFUSAL (the probe is discarded
  and sampling restarts from the prompt); else if |q| = L: REFUSAL (the probe
  reached the length cap while compatible);
* a compatible q with some pi, |pi| >= min_confirm, as a prefix stays
  compatible for every extension, so the outcome is REFUSAL from that token on
  ("confirmed"); the probe still runs to the stop token or to L to produce the
  returned text.

Decision codes: 0 = PENDING, 1 = REFUSAL, 2 = NON_REFUSAL.  ``decisive_step`` is
the 0-based index, in the probe's token stream, of the token at which the
outcome became known.  Pinned by the paper's worked examples
(tests/golden/gate_paper_examples.txt) and by hand-derived planted cases.
"""
from __future__ import annotations

import dataclasses
from typing import List, Sequence

import numpy as np

PENDING, REFUSAL, NON_REFUSAL = 0, 1, 2


def is_prefix(a: Sequence[int], b: Sequence[int]) -> bool:
    """True when sequence a is a prefix of sequence b (the empty sequence is a prefix of all)."""
    return len(a) <= len(b) and list(a) == list(b[:len(a)])


def compatible(q: Sequence[int], P: Sequence[Sequence[int]], min_confirm: int = 2) -> bool:
    """C(q, P) by a naive scan over the refusal list."""
    q = [int(x) for x in q]
    for pi in P:
        pi = [int(x) for x in pi]
        if is_prefix(q, pi):
            return True
        if len(pi) >= min_confirm and is_prefix(pi, q):
            return True
    return False


def confirmed(q: Sequence[int], P: Sequence[Sequence[int]], min_confirm: int = 2) -> bool:
    """Some pi with |pi| >= min_confirm is a prefix of q (q then stays compatible)."""
    q = [int(x) for x in q]
    return any(len(pi) >= min_confirm and is_prefix([int(x) for x in pi], q) for pi in P)


@dataclasses.dataclass
class GateState:
    q: List[int] = dataclasses.field(default_factory=list)
    steps: int = 0               # probe tokens consumed, stop token included
    decision: int = PENDING
    decisive_step: int = -1
    is_confirmed: bool = False
    done: bool = False           # the probe has ended (stop, cap, or discarded)


def gate_step(st: GateState, y: int, P, eos: int, max_len: int, min_confirm: int = 2) -> None:
    """Consume one greedy probe token y (in place)."""
    if st.done:
        return
    step = st.steps
    st.steps += 1
    if eos >= 0 and int(y) == eos:
        st.done = True
        if st.decision == PENDING:
            ok = compatible(st.q, P, min_confirm)
            st.decision = REFUSAL if ok else NON_REFUSAL
            st.decisive_step = step
        return
    st.q.append(int(y))
    if not compatible(st.q, P, min_confirm):
        # a confirmed probe can never get here: its confirming prefix stays a prefix
        st.decision = NON_REFUSAL
        st.decisive_step = step
        st.done = True
        return
    if not st.is_confirmed and confirmed(st.q, P, min_confirm):
        st.is_confirmed = True
        if st.decision == PENDING:
            st.decision = REFUSAL
            st.decisive_step = step
    if len(st.q) >= max_len:
        st.done = True
        if st.decision == PENDING:
            st.decision = REFUSAL
            st.decisive_step = step


def run_gate(tokens: np.ndarray, P, eos: int, max_len: int, min_confirm: int = 2,
             states: List[GateState] = None) -> List[GateState]:
    """Feed each group's probe tokens [groups, n] through :func:`gate_step`."""
    tokens = np.asarray(tokens)
    G = tokens.shape[0]
    if states is None:
        states = [GateState() for _ in range(G)]
    for g in range(G):
        for y in tokens[g]:
            gate_step(states[g], int(y), P, eos, max_len, min_confirm)
    return states


def row_mask_update(states: List[GateState], rows_per_group: int, row_active: np.ndarray) -> np.ndarray:
    """Rows a gate state switches off: the probe row once the probe has ended; the
    sample rows of a group whose outcome is REFUSAL (their draws are discarded)."""
    out = np.array(row_active, dtype=np.uint8, copy=True)
    for g, st in enumerate(states):
        if st.done:
            out[g * rows_per_group] = 0
        if st.decision == REFUSAL:
            out[g * rows_per_group + 1:(g + 1) * rows_per_group] = 0
    return out


def refusal_gated_decode(greedy_stream: Sequence[int], P, c: int, max_len: int, eos: int,
                         min_confirm: int = 2):
    """Alg. 1 as written, on a pre-drawn greedy token stream (G_M's outputs in order).

    Returns ("refusal", q) when the greedy probe is returned, or ("sample", q) when
    the method falls back to S_{T,theta}(M, p); q is the probe at that point.
    Used to check that the per-token gate above reaches Alg. 1's outcome.
    """
    it = iter(greedy_stream)
    q: List[int] = []

    def G_M():
        y = int(next(it))
        stop = eos >= 0 and y == eos
        return y, stop

    for _ in range(c):
        y, stop = G_M()
        if not stop:
            q.append(y)
        if not compatible(q, P, min_confirm):
            return "sample", q
        if stop or len(q) == max_len:
            return "refusal", q
    # B_M: continue greedy to the remaining budget; decisive event z
    while True:
        y, stop = G_M()
        if not stop:
            q.append(y)
        if not compatible(q, P, min_confirm):
            return "sample", q
        if stop or len(q) == max_len:
            return "refusal", q
