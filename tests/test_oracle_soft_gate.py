"""Pins of the soft compatibility gate oracle (the appendix ablation's Alg. 2).

Anchors: the appendix's worked illustration on a toy vocabulary
(tests/golden/soft_gate_example.txt, outcomes worked out by hand), the limits
that reduce it to the hard gate (K = 1, rho > 1, steps past the window c),
brute force over every compatible candidate, and the continue condition
(m >= rho with a non-empty A_ref) at an exactly representable m.
"""
import math
import os

import numpy as np
import pytest

from oracle import gate as ogate
from oracle import soft_gate as osg
from paper_2607_20791_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "soft_gate_example.txt")


def _golden():
    vocab, prefixes, cases, probs, eos = [], [], [], None, -1
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        kind, rest = line.split(" ", 1)
        if kind == "vocab":
            vocab = rest.split()
        elif kind == "eos":
            eos = vocab.index(rest)
        elif kind == "prefix":
            prefixes.append([vocab.index(t) for t in rest.split()])
        elif kind == "probs":
            probs = np.array([float(x) for x in rest.split()])
        else:
            lhs, rhs = rest.split(" -> ")
            kv = dict(f.split("=") for f in lhs.split())
            out = rhs.split()
            cases.append((int(kv["K"]), float(kv["rho"]), out[0], float(out[-1].split("=")[1])))
    return vocab, eos, prefixes, probs, cases


def test_paper_illustration():
    vocab, eos, P, probs, cases = _golden()
    assert abs(probs.sum() - 1.0) < 1e-12
    for k, rho, outcome, mass in cases:
        st = ogate.GateState()
        ogate.gate_step(st, vocab.index("I"), P, eos, 16)  # the partial probe "I"
        r = osg.soft_gate_step(st, np.log(probs), P, eos, 16, c=8, k=k, rho=rho)
        assert r.soft and abs(r.mass - mass) < 1e-12, (k, rho, r)
        if outcome == "discard":
            assert r.token is None and st.decision == ogate.NON_REFUSAL and st.done
            assert st.decisive_step == 1
        else:
            tok = outcome.split("=")[1]
            assert r.token == vocab.index(tok) and not st.done
            assert st.q == [vocab.index("I"), vocab.index(tok)]
            # "I cannot" is a whole refusal opening of two tokens: confirmed, so REFUSAL
            assert st.decision == (ogate.REFUSAL if ogate.confirmed(st.q, P) else ogate.PENDING)


def _random_case(seed, V=50, n_seq=6):
    P = workloads.make_refusal_set(n_seq, 2, 5, V, seed)
    rng = np.random.default_rng(seed)
    return P, rng


def test_reduces_to_the_hard_gate():
    for seed in range(20):
        P, rng = _random_case(seed)
        for trial in range(10):
            logits = rng.standard_normal(50) * 3
            pre = list(P[trial % len(P)][:rng.integers(0, 2)])
            for k, rho, c in ((1, 0.0, 8), (50, 1.5, 8), (50, 0.0, 0)):
                a, b = ogate.GateState(), ogate.GateState()
                for t in pre:
                    ogate.gate_step(a, int(t), P, -1, 16)
                    ogate.gate_step(b, int(t), P, -1, 16)
                r = osg.soft_gate_step(a, logits, P, -1, 16, c=c, k=k, rho=rho)
                y = int(np.argmax(logits))
                ogate.gate_step(b, y, P, -1, 16)
                # the same outcome; a discarded soft step does not append y to q
                assert (a.decision, a.done, a.decisive_step, a.steps) == (b.decision, b.done, b.decisive_step,
                                                                         b.steps), (seed, trial, k, rho, c)
                assert a.q == (b.q[:-1] if r.soft else b.q)
                assert r.token == (None if r.soft else y)


def test_brute_force_soft_choice():
    for seed in range(30):
        P, rng = _random_case(seed, V=40)
        logits = np.round(rng.standard_normal(40) * 2, 1)  # rounding plants ties
        st = ogate.GateState()
        r = osg.soft_gate_step(st, logits, P, -1, 16, c=4, k=12, rho=0.0)
        y = int(np.argmax(logits))
        if ogate.compatible([y], P):
            assert r.token == y and not r.soft
            continue
        p = np.exp(logits - logits.max())
        p /= p.sum()
        # brute force: the 12 best (value, then index), the compatible ones, their mass
        ranked = sorted(range(40), key=lambda i: (-logits[i], i))[:12]
        comp = [a for a in ranked if ogate.compatible([a], P)]
        assert r.a_ref == comp
        assert math.isclose(r.mass, sum(p[a] for a in comp), rel_tol=0, abs_tol=1e-12)
        if comp:
            assert r.token == comp[0] and st.q == [comp[0]]
        else:
            assert r.token is None and st.decision == ogate.NON_REFUSAL


def test_top_k_ties_and_softmax():
    l = np.array([1.0, 3.0, 3.0, 2.0, 3.0])
    assert list(osg.top_k(l, 3)) == [1, 2, 4]
    p = osg.softmax(np.log(np.array([0.1, 0.2, 0.7])))
    assert np.allclose(p, [0.1, 0.2, 0.7], atol=1e-15)


def test_mass_threshold_is_inclusive_and_needs_a_candidate():
    # Alg. 2 goes on when m >= rho and A_ref is not empty.  Four equal logits give
    # p = 1/4 exactly in fp64; the greedy token 0 leaves the refusal set, tokens 1
    # and 2 keep it, so m = 1/2 exactly.
    P = [[1, 3], [2, 3]]
    logits = np.zeros(4)
    st = ogate.GateState()
    r = osg.soft_gate_step(st, logits, P, -1, 8, c=2, k=4, rho=0.5)
    assert r.soft and r.mass == 0.5 and r.a_ref == [1, 2] and r.token == 1 and not st.done
    st = ogate.GateState()
    r = osg.soft_gate_step(st, logits, P, -1, 8, c=2, k=4, rho=float(np.nextafter(0.5, 1.0)))
    assert r.soft and r.token is None and st.done and st.decision == ogate.NON_REFUSAL
    # rho = 0 with no compatible token in the top K: A_ref is empty, so the probe ends
    st = ogate.GateState()
    r = osg.soft_gate_step(st, logits, P, -1, 8, c=2, k=1, rho=0.0)
    assert r.soft and r.a_ref == [] and r.mass == 0.0 and r.token is None and st.done
