"""The tiny configuration's 16-step gated loop end to end on the GPU: attention,
sample head and trie gate per step, with the gate's row mask fed back into the
next step, against the oracle run the same way."""
import numpy as np
import pytest

from oracle import attention as oattn
from oracle import gate as ogate
from oracle import sampling as osamp
from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_tiny_sixteen_step_loop(gpu_lib, seed):
    import torch
    first = workloads.tiny(seed=seed, step=0)
    G, rpg = first.attn.num_groups, first.attn.rows_per_group
    P, eos, L = first.gate.refusal_seqs, first.gate.eos, first.gate.max_len
    trie = binding.Trie(P, 2)
    st = binding.new_gate_state(G)
    binding.rgd_gate_state_init(st, G)
    row_active = torch.ones(G * rpg, dtype=torch.uint8, device="cuda")
    ref_states = [ogate.GateState() for _ in range(G)]
    ref_active = np.ones(G * rpg, np.uint8)
    for step in range(16):
        case = workloads.tiny(seed=seed, step=step)
        case.attn.row_active = ref_active.copy()
        case.head.row_active = ref_active.copy()
        att = device.attn_to_device(case.attn)
        att.row_active = row_active
        head = device.head_to_device(case.head)
        head.row_active = row_active
        att.run()
        head.run(with_mask=False)
        binding.rgd_probe_gate(trie, G, rpg, head.token_out, 1, rpg, eos, L, st, row_active, head.dev_status)
        torch.cuda.synchronize()
        # oracle: same step
        ref_o, _ = oattn.decode_attention_case(case.attn)
        o = att.out.float().cpu().numpy()
        for r in range(G * rpg):
            if ref_active[r]:
                assert np.all(np.abs(o[r] - ref_o[r]) <= 2e-3 + 1e-2 * np.abs(ref_o[r])), (step, r)
        ref_h = osamp.sample_head(case.head.logits, "f32", case.head.is_probe, case.head.temperature,
                                  case.head.min_p, case.head.seed, case.head.step, ref_active)
        tok = head.token_out.cpu().numpy()
        for r in range(G * rpg):
            assert tok[r] == ref_h.tokens[r] or ref_h.boundary[r], (step, r)
        for g in range(G):
            if ref_active[g * rpg]:
                ogate.gate_step(ref_states[g], int(ref_h.tokens[g * rpg]), P, eos, L)
        ref_active = ogate.row_mask_update(ref_states, rpg, ref_active)
        assert np.array_equal(row_active.cpu().numpy(), ref_active), step
        got = binding.decode_gate_state(st)
        assert got["decision"][0] == ref_states[0].decision
        assert got["decisive_step"][0] == ref_states[0].decisive_step
        assert int(att.dev_status.item()) == 0 and int(head.dev_status.item()) == 0
    trie.close()


@pytest.mark.parametrize("seed", [0, 1])
def test_tiny_sixteen_step_loop_in_one_graph(gpu_lib, seed):
    """The whole 16-step probe loop (attention, sample head, trie gate per step,
    the gate's row mask feeding the next step) captured as ONE CUDA graph and
    replayed: every step's tokens and the final gate state against the oracle
    run the same way."""
    import torch
    steps = 16
    first = workloads.tiny(seed=seed, step=0)
    G, rpg = first.attn.num_groups, first.attn.rows_per_group
    P, eos, L = first.gate.refusal_seqs, first.gate.eos, first.gate.max_len
    trie = binding.Trie(P, 2)
    st = binding.new_gate_state(G)
    row_active = torch.ones(G * rpg, dtype=torch.uint8, device="cuda")
    cases = [workloads.tiny(seed=seed, step=s) for s in range(steps)]
    atts, heads = [], []
    for case in cases:  # every step's inputs and outputs resident before capture
        a = device.attn_to_device(case.attn)
        a.row_active = row_active
        h = device.head_to_device(case.head)
        h.row_active = row_active
        atts.append(a)
        heads.append(h)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for a, h in zip(atts[:1], heads[:1]):  # warm-up outside capture (kernel attributes)
            a.run(stream=stream.cuda_stream)
            h.run(stream=stream.cuda_stream, with_mask=False)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            binding.rgd_gate_state_init(st, G, stream=stream.cuda_stream)
            row_active.fill_(1)
            for a, h in zip(atts, heads):
                a.run(stream=stream.cuda_stream)
                h.run(stream=stream.cuda_stream, with_mask=False)
                binding.rgd_probe_gate(trie, G, rpg, h.token_out, 1, rpg, eos, L, st, row_active, h.dev_status,
                                       stream=stream.cuda_stream)
        graph.replay()
        torch.cuda.synchronize()
    # the oracle, step by step with its own row mask
    ref_states = [ogate.GateState() for _ in range(G)]
    ref_active = np.ones(G * rpg, np.uint8)
    for s, (case, h) in enumerate(zip(cases, heads)):
        ref_h = osamp.sample_head(case.head.logits, "f32", case.head.is_probe, case.head.temperature,
                                  case.head.min_p, case.head.seed, case.head.step, ref_active)
        tok = h.token_out.cpu().numpy()
        for r in range(G * rpg):
            assert tok[r] == ref_h.tokens[r] or ref_h.boundary[r], (s, r)
        for g in range(G):
            if ref_active[g * rpg]:
                ogate.gate_step(ref_states[g], int(ref_h.tokens[g * rpg]), P, eos, L)
        ref_active = ogate.row_mask_update(ref_states, rpg, ref_active)
    assert np.array_equal(row_active.cpu().numpy(), ref_active)
    got = binding.decode_gate_state(st)
    for g in range(G):
        assert got["decision"][g] == ref_states[g].decision
        assert got["decisive_step"][g] == ref_states[g].decisive_step
    trie.close()
