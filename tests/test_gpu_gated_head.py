"""The sample head with the hard gate fused in (rgd_sample_head_gated) and the
one-call decode step (rgd_decode_step) on the GPU.

The fused kernel must give exactly what the two separate calls give (tokens,
kept counts, gate states and row masks bit for bit), and both agree with the
oracle: the head's tokens (bit-exact outside boundary rows), the gate's
decisions and decisive steps on the probe tokens (bit-exact), attention within
|gpu - ref| <= 2e-3 + 1e-2 |ref|."""
import numpy as np
import pytest

from oracle import attention as oattn
from oracle import gate as ogate
from oracle import sampling as osamp
from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu


def _run_both(head_case, gate_case, rpg):
    """Separate calls (head, then gate) and the fused call on the same inputs,
    from the same gate state and row mask; returns both results."""
    import torch
    G = head_case.rows // rpg
    trie = binding.Trie(gate_case.refusal_seqs, gate_case.min_confirm)
    out = []
    for fused in (False, True):
        dev = device.head_to_device(head_case)
        st = binding.new_gate_state(G)
        binding.rgd_gate_state_init(st, G)
        ra = dev.row_active.clone()
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        if fused:
            binding.rgd_sample_head_gated(dev.logits, dev.is_probe, dev.temperature, dev.min_p, dev.seed,
                                          dev.step, ra, dev.token_out, dev.kept_count, trie, rpg, gate_case.eos,
                                          gate_case.max_len, st, status)
        else:
            binding.rgd_sample_head(dev.logits, dev.is_probe, dev.temperature, dev.min_p, dev.seed, dev.step, ra,
                                    dev.token_out, dev.kept_count, None, status)
            binding.rgd_probe_gate(trie, G, rpg, dev.token_out, 1, rpg, gate_case.eos, gate_case.max_len, st, ra,
                                   status)
        torch.cuda.synchronize()
        out.append({"tok": dev.token_out.cpu().numpy(), "cnt": dev.kept_count.cpu().numpy(),
                    "state": st.cpu().numpy(), "ra": ra.cpu().numpy(), "status": int(status.item())})
    trie.close()
    return out


def _check_against_oracle(head_case, gate_case, rpg, res):
    ref = osamp.sample_head(head_case.logits, head_case.dtype, head_case.is_probe, head_case.temperature,
                            head_case.min_p, head_case.seed, head_case.step, head_case.row_active)
    for r in range(head_case.rows):
        assert res["tok"][r] == ref.tokens[r] or ref.boundary[r], r
    G = head_case.rows // rpg
    probe = np.array([[ref.tokens[g * rpg]] for g in range(G)], np.int32)
    want = ogate.run_gate(probe, gate_case.refusal_seqs, gate_case.eos, gate_case.max_len, gate_case.min_confirm)
    import torch
    got = binding.decode_gate_state(torch.from_numpy(res["state"]))
    for g, s in enumerate(want):
        assert got["decision"][g] == s.decision and got["decisive_step"][g] == s.decisive_step, g
    assert np.array_equal(res["ra"], ogate.row_mask_update(want, rpg, head_case.row_active))


@pytest.mark.parametrize("name", ["tiny", "llama8b", "long_prompt", "high_batch"])
def test_fused_equals_separate_calls(gpu_lib, name):
    case = workloads.CONFIGS[name](seed=3, **({} if name == "tiny" else {"with_kv": False}))
    rpg = case.attn.rows_per_group
    sep, fus = _run_both(case.head, case.gate, rpg)
    for k in ("tok", "cnt", "state", "ra"):
        assert np.array_equal(sep[k], fus[k]), k
    assert sep["status"] == fus["status"] == 0
    # the reserved byte (the fused kernel's row count) is back at zero
    assert np.all(fus["state"].reshape(-1, binding.GATE_STATE_BYTES)[:, 19] == 0)
    _check_against_oracle(case.head, case.gate, rpg, fus)


def test_fused_planted_probes_many_steps(gpu_lib):
    """Groups whose probe row argmax follows planted streams (refusal sequences,
    divergences, the stop token): 24 fused calls from one state, against the
    separate calls and the oracle's gate, step by step."""
    import torch
    G, rpg, V, steps = 40, 3, 5000, 24
    eos = V - 1
    seqs = workloads.make_refusal_set(30, 2, 6, V, seed=4, avoid=[eos])
    streams = workloads.loop_probe_streams(seqs, G, steps, V, seed=4, eos=eos)
    gate = workloads.GateCase(name="planted", refusal_seqs=seqs, tokens=streams, eos=eos, max_len=12,
                              rows_per_group=rpg)
    trie = binding.Trie(seqs, 2)
    st = [binding.new_gate_state(G) for _ in range(2)]
    for s in st:
        binding.rgd_gate_state_init(s, G)
    ra = [torch.ones(G * rpg, dtype=torch.uint8, device="cuda") for _ in range(2)]
    ref_states = [ogate.GateState() for _ in range(G)]
    ref_ra = np.ones(G * rpg, np.uint8)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    base = workloads.zipf_logits(G * rpg, V, seed=5)
    for t in range(steps):
        logits = base.copy()
        logits[np.arange(G) * rpg, streams[:, t]] = 64.0  # the probe's greedy token this step
        case = workloads.make_head_case("planted", logits, "f32", np.tile([1] + [0] * (rpg - 1), G),
                                        np.tile([0.0] + [1.5] * (rpg - 1), G), [0.1] * (G * rpg), seed=6, step=t)
        dev = device.head_to_device(case)
        tok = []
        for fused in (False, True):
            if fused:
                binding.rgd_sample_head_gated(dev.logits, dev.is_probe, dev.temperature, dev.min_p, dev.seed, t,
                                              ra[1], dev.token_out, dev.kept_count, trie, rpg, eos, gate.max_len,
                                              st[1], status)
            else:
                binding.rgd_sample_head(dev.logits, dev.is_probe, dev.temperature, dev.min_p, dev.seed, t, ra[0],
                                        dev.token_out, dev.kept_count, None, status)
                binding.rgd_probe_gate(trie, G, rpg, dev.token_out, 1, rpg, eos, gate.max_len, st[0], ra[0],
                                       status)
            torch.cuda.synchronize()
            tok.append(dev.token_out.cpu().numpy().copy())
        assert np.array_equal(tok[0], tok[1]), t
        assert torch.equal(st[0], st[1]) and torch.equal(ra[0], ra[1]), t
        for g in range(G):
            if ref_ra[g * rpg]:
                assert tok[1][g * rpg] == streams[g, t]
                ogate.gate_step(ref_states[g], int(streams[g, t]), seqs, eos, gate.max_len)
            else:
                assert tok[1][g * rpg] == -1
        ref_ra = ogate.row_mask_update(ref_states, rpg, ref_ra)
        assert np.array_equal(ra[1].cpu().numpy(), ref_ra), t
    got = binding.decode_gate_state(st[1])
    for g, s in enumerate(ref_states):
        assert got["decision"][g] == s.decision and got["decisive_step"][g] == s.decisive_step, g
        assert got["done"][g] == int(s.done) and got["length"][g] == len(s.q), g
    assert {s.decision for s in ref_states} == {ogate.REFUSAL, ogate.NON_REFUSAL}
    assert int(status.item()) == 0
    trie.close()


def test_fused_inactive_probe_reports_bad_token(gpu_lib):
    """A probe row switched off while its probe has not ended gives the gate a
    -1 token: both forms skip it and set RGD_DEV_BAD_TOKEN."""
    case = workloads.tiny(seed=1)
    head = case.head
    head.row_active = np.array([0, 1, 1], np.uint8)
    sep, fus = _run_both(head, case.gate, 3)
    for k in ("tok", "cnt", "state", "ra"):
        assert np.array_equal(sep[k], fus[k]), k
    assert sep["status"] == fus["status"] == binding.RGD_DEV_BAD_TOKEN


def test_decode_step_one_call(gpu_lib):
    """rgd_decode_step on the Llama-3-8B-shaped step: attention against the
    oracle, tokens and gate against the separate calls."""
    import torch
    case = workloads.llama8b(seed=4)
    G, rpg = case.attn.num_groups, case.attn.rows_per_group
    att = device.attn_to_device(case.attn)
    head = device.head_to_device(case.head)
    trie = binding.Trie(case.gate.refusal_seqs, 2)
    st = binding.new_gate_state(G)
    binding.rgd_gate_state_init(st, G)
    ra = att.row_active.clone()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    binding.rgd_decode_step(att.shape, att.q, att.k_pages, att.v_pages, att.prompt_block_table, att.prompt_len,
                            att.suffix_block_table, att.suffix_len, att.softmax_scale, att.out, att.lse,
                            att.workspace, head.logits, head.is_probe, head.temperature, head.min_p, head.seed,
                            head.step, ra, head.token_out, head.kept_count, trie, case.gate.eos,
                            case.gate.max_len, st, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref_o, _ = oattn.decode_attention_case(case.attn)
    o = att.out.float().cpu().numpy()
    assert np.all(np.abs(o - ref_o) <= 2e-3 + 1e-2 * np.abs(ref_o))
    sep, _ = _run_both(case.head, case.gate, rpg)
    assert np.array_equal(head.token_out.cpu().numpy(), sep["tok"])
    assert np.array_equal(st.cpu().numpy(), sep["state"])
    assert np.array_equal(ra.cpu().numpy(), sep["ra"])
    trie.close()


def test_decode_step_rejects_before_launching(gpu_lib):
    """A bad head argument is refused before the attention is launched: the
    output stays untouched."""
    import torch
    case = workloads.tiny(seed=0)
    att = device.attn_to_device(case.attn)
    head = device.head_to_device(case.head)
    trie = binding.Trie(case.gate.refusal_seqs, 2)
    st = binding.new_gate_state(1)
    before = att.out.clone()
    with pytest.raises(binding.RgdError) as ei:
        binding.rgd_decode_step(att.shape, att.q, att.k_pages, att.v_pages, att.prompt_block_table,
                                att.prompt_len, att.suffix_block_table, att.suffix_len, att.softmax_scale, att.out,
                                att.lse, att.workspace, head.logits, head.is_probe, head.temperature, head.min_p,
                                head.seed, head.step, att.row_active, head.token_out, head.kept_count, trie,
                                case.gate.eos, 0, st)  # max_len 0
    assert ei.value.code == binding.RGD_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert torch.equal(att.out, before)
    trie.close()
