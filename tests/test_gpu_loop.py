"""The whole gated decode loop on the Llama-3-8B shape as ONE CUDA graph (Alg. 1,
with the probe and the sample rows of each prompt decoding side by side).

128 steps, each one rgd_decode_step (shared-prefix attention, then the sample
head with the hard gate fused in) from the prompt end: every active row appends
its token to its own suffix, the greedy probes follow planted streams (refusal
sequences in full, then to the length cap L = 128 or to the stop token;
divergences; random starts; a proper prefix, then the stop token).  Checked
against the oracle run the same way: every step's tokens (probe tokens
bit-exact, sampled tokens bit-exact outside boundary rows), the row masks, the
final gate states, each group's outcome and returned probe against Alg. 1 as
written (oracle.gate.refusal_gated_decode), and attention at four steps."""
import numpy as np
import pytest

from oracle import attention as oattn
from oracle import gate as ogate
from oracle import sampling as osamp
from paper_2607_20791_gb300 import binding, device, workloads

from conftest import report

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

ATTN_STEPS = (0, 1, 63, 127)


def _oracle_loop(case):
    """The oracle run the same way: per step the sample head on the step's
    logits over the active rows, the gate on the probe tokens, the row mask."""
    G, rpg, n = case.attn.num_groups, case.attn.rows_per_group, case.n_steps
    R = G * rpg
    states = [ogate.GateState() for _ in range(G)]
    active = np.ones(R, np.uint8)
    slen = np.zeros(R, np.int32)
    hist = []
    h = case.head
    for t in range(n):
        logits = workloads.loop_step_logits(case, t)
        res = osamp.sample_head(logits, "f32", h.is_probe, h.temperature, h.min_p, h.seed, t, active)
        hist.append({"active": active.copy(), "slen": slen.copy(), "res": res})
        for g in range(G):
            if active[g * rpg]:
                ogate.gate_step(states[g], int(res.tokens[g * rpg]), case.refusal_seqs, case.eos, case.max_len)
        slen = slen + active
        active = ogate.row_mask_update(states, rpg, active)
    return states, active, hist


def test_llama8b_gated_loop_in_one_graph(gpu_lib):
    import torch
    case = workloads.llama8b_loop(seed=0)
    G, rpg, n = case.attn.num_groups, case.attn.rows_per_group, case.n_steps
    loop = device.DeviceLoop(case, torch.cuda.Stream())
    loop.capture()
    loop.tok.fill_(-7)
    loop.graph.replay()
    torch.cuda.synchronize()
    assert int(loop.status.item()) == 0
    tok = loop.tok.cpu().numpy()
    states, active, hist = _oracle_loop(case)
    boundary = mismatched = 0
    for t, hs in enumerate(hist):
        res = hs["res"]
        for r in range(G * rpg):
            if not hs["active"][r]:
                assert tok[t, r] == -1, (t, r)
            elif tok[t, r] != res.tokens[r]:
                assert res.boundary[r], (t, r, tok[t, r], res.tokens[r])
                mismatched += 1
            boundary += int(hs["active"][r] and res.boundary[r])
    assert mismatched <= max(1, boundary // 10)
    assert np.array_equal(loop.row_active.cpu().numpy(), active)
    assert np.array_equal(loop.suffix_len.cpu().numpy(), hist[-1]["slen"] + hist[-1]["active"])
    got = binding.decode_gate_state(loop.state)
    outcomes = []
    for g, s in enumerate(states):
        assert got["decision"][g] == s.decision and got["decisive_step"][g] == s.decisive_step, g
        assert got["done"][g] == int(s.done) and got["length"][g] == len(s.q), g
        assert got["confirmed"][g] == int(s.is_confirmed), g
        # Alg. 1 as written, on the same greedy stream: the same outcome, and a
        # returned refusal is the probe the gate kept
        kind, q = ogate.refusal_gated_decode(case.probe_streams[g], case.refusal_seqs, case.gate_cap,
                                             case.max_len, case.eos)
        assert kind == ("refusal" if s.decision == ogate.REFUSAL else "sample"), g
        if kind == "refusal":
            assert got["length"][g] == len(q) and list(case.probe_streams[g][:len(q)]) == q, g
        outcomes.append(kind)
        # a refused group's sample rows stop at its decisive step; a non-refused
        # group's sample rows decode every step from the prompt (their suffix
        # never holds the probe's tokens)
        for i in range(1, rpg):
            r = g * rpg + i
            drew = tok[:, r] >= 0
            if s.decision == ogate.REFUSAL:
                assert drew[:s.decisive_step + 1].all() and not drew[s.decisive_step + 1:].any(), (g, i)
            else:
                assert drew.all(), (g, i)
    assert set(outcomes) == {"refusal", "sample"}
    report(f"llama8b gated loop: {n} steps, outcomes {outcomes.count('refusal')} refusal / "
           f"{outcomes.count('sample')} sample, {boundary} boundary draws, {mismatched} boundary mismatches")
    # attention at a few steps, with that step's suffix lengths and row mask
    out = loop.out.float().cpu().numpy()
    for t in ATTN_STEPS:
        a = case.attn
        a.suffix_len = hist[t]["slen"].astype(np.int32)
        a.row_active = hist[t]["active"]
        rows = [r for r in range(G * rpg) if hist[t]["active"][r]]
        ref_o, _ = oattn.decode_attention_case(a, rows=rows)
        for r in rows:
            err = np.abs(out[t, r] - ref_o[r])
            assert np.all(err <= 2e-3 + 1e-2 * np.abs(ref_o[r])), (t, r, float(err.max()))
    loop.close()
