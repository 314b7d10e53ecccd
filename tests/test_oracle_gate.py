"""Pins of the oracle's compatibility predicate and hard gate.

Anchors: the paper's worked text examples (tests/golden/gate_paper_examples.txt,
on a toy word-level vocabulary), Alg. 1 run literally on token streams, and
hand-derived planted probes.
"""
import os

import numpy as np

from oracle import gate
from paper_2607_20791_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "gate_paper_examples.txt")


def _load_golden():
    prefixes, probes, streams = [], [], []
    for line in open(GOLDEN):
        line = line.rstrip("\n")
        if not line.strip() or line.startswith("#"):
            continue
        kind, rest = line.split(" ", 1)
        if kind == "prefix":
            prefixes.append(rest.split())
        else:
            toks, fields = rest.split(" | ")
            kv = dict(f.split("=") for f in fields.split())
            (probes if kind == "probe" else streams).append((toks.split(), kv))
    return prefixes, probes, streams


def _vocab(prefixes, probes, streams):
    words = {"<eos>": 0}
    for seq in prefixes + [p[0] for p in probes] + [s[0] for s in streams]:
        for w in seq:
            words.setdefault(w, len(words))
    return words


def test_paper_examples_predicate():
    prefixes, probes, streams = _load_golden()
    vocab = _vocab(prefixes, probes, streams)
    P = [[vocab[w] for w in p] for p in prefixes]
    assert len(probes) >= 5
    for toks, kv in probes:
        q = [vocab[w] for w in toks]
        assert gate.compatible(q, P) == bool(int(kv["compatible"])), toks
        assert gate.confirmed(q, P) == bool(int(kv["confirmed"])), toks


def test_paper_examples_streams():
    prefixes, probes, streams = _load_golden()
    vocab = _vocab(prefixes, probes, streams)
    P = [[vocab[w] for w in p] for p in prefixes]
    eos = vocab["<eos>"]
    for toks, kv in streams:
        stream = [vocab[w] for w in toks]
        outcome, _ = gate.refusal_gated_decode(stream + [eos] * 4, P, c=3, max_len=128, eos=eos)
        assert outcome == kv["outcome"], toks
        st = gate.run_gate(np.array([stream]), P, eos=eos, max_len=128)[0]
        want = gate.REFUSAL if kv["outcome"] == "refusal" else gate.NON_REFUSAL
        assert st.decision == want and st.decisive_step == int(kv["at"]), (toks, st)


def test_two_token_minimum():
    P = [[5], [7, 8]]
    assert gate.compatible([5], P)            # q is a prefix of (equal to) pi = [5]
    assert not gate.compatible([5, 1], P)     # [5] is a prefix of q, but |pi| = 1 < 2
    assert gate.compatible([5, 1], P, min_confirm=1)
    assert gate.compatible([7, 8, 9, 9], P) and gate.confirmed([7, 8, 9], P)
    assert not gate.confirmed([5, 9], P)


def test_empty_probe_and_empty_set():
    assert gate.compatible([], [[1, 2]])
    assert not gate.compatible([], [])
    st = gate.run_gate(np.array([[3, 4]]), [], eos=-1, max_len=8)[0]
    assert st.decision == gate.NON_REFUSAL and st.decisive_step == 0
    st = gate.run_gate(np.array([[0]]), [], eos=0, max_len=8)[0]   # stop first, P empty
    assert st.decision == gate.NON_REFUSAL and st.decisive_step == 0
    st = gate.run_gate(np.array([[0]]), [[1, 2]], eos=0, max_len=8)[0]  # stop first
    assert st.decision == gate.REFUSAL and st.decisive_step == 0 and st.q == []


def test_planted_probes_hand_derived():
    P = [[1, 2, 3], [1, 2, 3, 4, 5], [9, 9], [1, 7]]
    cases = [
        # (stream, eos, L) -> (decision, decisive_step, done, |q|)
        (([1, 2, 3, 6, 6, 6], -1, 6), (gate.REFUSAL, 2, True, 6)),      # confirm at 3rd token
        (([1, 2, 6, 6], -1, 8), (gate.NON_REFUSAL, 2, True, 3)),        # diverge mid-way
        (([1, 2, 3, 4], -1, 4), (gate.REFUSAL, 2, True, 4)),            # confirmed, then cap
        (([1, 2], -1, 2), (gate.REFUSAL, 1, True, 2)),                  # proper prefix until L
        (([1, 2, 0], 0, 8), (gate.REFUSAL, 2, True, 2)),                # stop while pending
        (([4, 1, 2], -1, 8), (gate.NON_REFUSAL, 0, True, 1)),           # random start
        (([9, 9, 1], -1, 8), (gate.REFUSAL, 1, False, 3)),              # confirmed, still running
        (([1, 7, 0, 5], 0, 8), (gate.REFUSAL, 1, True, 2)),             # confirmed then stop
        (([1], -1, 8), (gate.PENDING, -1, False, 1)),                   # undecided
    ]
    for (stream, eos, L), (dec, at, done, qlen) in cases:
        st = gate.run_gate(np.array([stream]), P, eos=eos, max_len=L)[0]
        assert (st.decision, st.decisive_step, st.done, len(st.q)) == (dec, at, done, qlen), stream


def test_duplicates_and_nested_sequences():
    P = [[1, 2, 3, 4], [1, 2, 3, 4], [1, 2]]
    st = gate.run_gate(np.array([[1, 2, 5]]), P, eos=-1, max_len=8)[0]
    assert st.decision == gate.REFUSAL and st.decisive_step == 1 and not st.done


def test_gate_matches_algorithm_1_on_planted_streams():
    # the per-token gate and Alg. 1 run literally agree on outcome for every c
    case = workloads.gate_sweep(groups=128, n_seq=50, vocab=64, n_steps=16, seed=4, eos=63)
    for g in range(case.groups):
        stream = [int(x) for x in case.tokens[g]]
        st = gate.run_gate(np.array([stream]), case.refusal_seqs, eos=63, max_len=12)[0]
        for c in (1, 3, 12):
            if st.decision == gate.PENDING:
                continue  # stream too short for Alg. 1 to finish
            outcome, _ = gate.refusal_gated_decode(stream, case.refusal_seqs, c, 12, 63)
            assert outcome == ("refusal" if st.decision == gate.REFUSAL else "sample")


def test_row_mask_update():
    P = [[1, 2]]
    sts = gate.run_gate(np.array([[1, 2], [5, 5], [1, 1]]), P, eos=-1, max_len=8)
    mask = gate.row_mask_update(sts, 3, np.ones(9, np.uint8))
    # group 0 confirmed (REFUSAL, probe still running): samples off
    # group 1 NON_REFUSAL: probe off; group 2 NON_REFUSAL at step 1: probe off
    assert mask.tolist() == [1, 0, 0, 0, 1, 1, 0, 1, 1]
