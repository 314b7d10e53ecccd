"""Trie gate on the GPU vs the oracle's naive scan: decisions, decisive steps,
confirmation and row masks bit-exact."""
import numpy as np
import pytest

from oracle import gate as ogate
from paper_2607_20791_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


def _gpu_gate(seqs, tokens, eos, max_len, rpg=1, min_confirm=2, per_token=False, row_active=None):
    import torch
    G, n = tokens.shape
    trie = binding.Trie(seqs, min_confirm)
    st = binding.new_gate_state(G)
    binding.rgd_gate_state_init(st, G)
    tok = torch.from_numpy(np.ascontiguousarray(tokens, dtype=np.int32)).cuda()
    ra = torch.from_numpy(np.ones(G * rpg, np.uint8) if row_active is None else row_active).cuda()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    if per_token:
        for k in range(n):
            binding.rgd_probe_gate(trie, G, rpg, tok.data_ptr() + 4 * k, 1, n, eos, max_len, st, ra, status)
    else:
        binding.rgd_probe_gate(trie, G, rpg, tok, n, n, eos, max_len, st, ra, status)
    torch.cuda.synchronize()
    out = binding.decode_gate_state(st)
    trie.close()
    return out, ra.cpu().numpy(), int(status.item())


def _compare(seqs, tokens, eos, max_len, rpg=1, min_confirm=2, per_token=False):
    got, ra, status = _gpu_gate(seqs, tokens, eos, max_len, rpg, min_confirm, per_token)
    ref = ogate.run_gate(tokens, seqs, eos, max_len, min_confirm)
    assert status == 0
    for g, st in enumerate(ref):
        assert got["decision"][g] == st.decision, (g, got["decision"][g], st)
        assert got["decisive_step"][g] == st.decisive_step, g
        assert got["done"][g] == int(st.done), g
        assert got["confirmed"][g] == int(st.is_confirmed), g
        assert got["length"][g] == len(st.q), g
        assert got["steps"][g] == st.steps, g
    want = ogate.row_mask_update(ref, rpg, np.ones(len(ref) * rpg, np.uint8))
    assert np.array_equal(ra, want)
    return ref


@pytest.mark.parametrize("per_token", [False, True])
def test_gate_sweep_full_size(gpu_lib, per_token):
    case = workloads.gate_sweep(groups=1024, n_seq=1000, vocab=128256, n_steps=32, seed=3)
    ref = _compare(case.refusal_seqs, case.tokens, case.eos, case.max_len, per_token=per_token)
    kinds = {st.decision for st in ref}
    assert kinds == {ogate.REFUSAL, ogate.NON_REFUSAL}


def test_gate_with_stop_token_and_rows(gpu_lib):
    case = workloads.gate_sweep(groups=300, n_seq=200, vocab=500, n_steps=20, seed=9, eos=499)
    _compare(case.refusal_seqs, case.tokens, case.eos, 12, rpg=5)
    _compare(case.refusal_seqs, case.tokens, case.eos, 12, rpg=5, per_token=True)


def test_gate_edge_cases(gpu_lib):
    P = [[1, 2, 3], [1, 2, 3, 4, 5], [9, 9], [1, 7], [5]]
    toks = np.array([
        [1, 2, 3, 6, 6, 6], [1, 2, 6, 6, 0, 0], [1, 2, 3, 4, 0, 0], [1, 2, 0, 7, 7, 7],
        [4, 1, 2, 0, 0, 0], [9, 9, 1, 1, 1, 1], [1, 7, 0, 5, 5, 5], [5, 1, 1, 1, 1, 1],
        [0, 1, 2, 3, 4, 5], [5, 0, 0, 0, 0, 0]], np.int32)
    for L in (1, 2, 4, 6, 8):
        for mc in (1, 2, 3):
            _compare(P, toks, 0, L, min_confirm=mc)
            _compare(P, toks, -1, L, min_confirm=mc, per_token=True)


def test_empty_refusal_set(gpu_lib):
    toks = np.array([[3, 4], [0, 1]], np.int32)
    _compare([], toks, 0, 8)


def test_negative_tokens_are_reported(gpu_lib):
    got, _, status = _gpu_gate([[1, 2]], np.array([[1, -5, 2]], np.int32), -1, 8)
    assert status & binding.RGD_DEV_BAD_TOKEN
    assert got["decision"][0] == binding.RGD_REFUSAL and got["length"][0] == 2
