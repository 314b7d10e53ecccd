"""The soft compatibility gate (the appendix ablation's Alg. 2) on the GPU
against the fp64 oracle, step by step: appended token, decision, decisive step
and mass m.  The top-K membership is exact (comparisons of the same fp32
logits); m is an fp32 sum, so the continue/discard decision may differ only
when the exact m lies within 2e-5 relative of rho (counted, must be rare).
"""
import numpy as np
import pytest

from oracle import gate as ogate
from oracle import soft_gate as osg
from paper_2607_20791_gb300 import binding, workloads

pytestmark = pytest.mark.gpu

GOLDEN_VOCAB = "I think cannot can't 'm sorry the <eos>".split()


def _children(P, q):
    """Tokens that extend q along some refusal sequence (the trie children)."""
    out = set()
    for pi in P:
        pi = [int(x) for x in pi]
        if len(pi) > len(q) and pi[:len(q)] == list(q):
            out.add(pi[len(q)])
    return sorted(out)


def _plant(rng, logits, P, states, eos, boost_frac=0.6):
    """Make the greedy token leave the refusal set while some compatible tokens
    keep probability, for a fraction of the groups (test inputs only)."""
    for g, st in enumerate(states):
        if st.done or rng.random() > boost_frac:
            continue
        kids = [a for a in _children(P, st.q) if a != eos]
        if not kids:
            continue
        top = float(logits[g].max())
        for a in rng.choice(kids, size=min(len(kids), 3), replace=False):
            logits[g, a] = top - float(rng.uniform(0.1, 2.5))
    return logits


def _run_loop(P, eos, groups, vocab, steps, c, k, rho, max_len, seed, dtype="f32", boost=0.6, scale=3.0):
    import torch
    rng = np.random.default_rng(seed)
    trie = binding.Trie(P, 2)
    st = binding.new_gate_state(groups)
    binding.rgd_gate_state_init(st, groups)
    rpg = 2
    active = torch.ones(groups * rpg, dtype=torch.uint8, device="cuda")
    tok = torch.empty(groups, dtype=torch.int32, device="cuda")
    mass = torch.empty(groups, dtype=torch.float32, device="cuda")
    ref = [ogate.GateState() for _ in range(groups)]
    ref_active = np.ones(groups * rpg, np.uint8)
    boundary = soft = deep = 0
    for step in range(steps):
        l32 = (rng.standard_normal((groups, vocab)) * scale).astype(np.float32)
        l32 = np.round(l32, 1)  # ties
        l32 = _plant(rng, l32, P, ref, eos, boost)
        full = np.zeros((groups * rpg, vocab), np.float32)
        full[::rpg] = l32  # the probe rows of the step's logits
        if dtype == "bf16":
            bits = workloads.f32_to_bf16_bits(full)
            full = (bits.astype(np.uint32) << 16).view(np.float32)
            dev = torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
        else:
            dev = torch.from_numpy(full).cuda()
        binding.rgd_soft_gate(trie, groups, rpg, dev, rpg * vocab, k, rho, c, eos, max_len, st, tok,
                              row_active=active, mass_out=mass)
        torch.cuda.synchronize()
        got = binding.decode_gate_state(st)
        t_gpu, m_gpu = tok.cpu().numpy(), mass.cpu().numpy()
        for g in range(groups):
            was_done = ref[g].done
            r = osg.soft_gate_step(ref[g], full[g * rpg].astype(np.float64), P, eos, max_len, c, k, rho)
            if was_done:
                assert t_gpu[g] == -1
                continue
            if r.soft:
                soft += 1
                # more than the four candidates the kernel's one pass ranks are
                # inside the top K: the kernel sorts them and searches the rest
                deep += len(r.a_ref) > 4
                assert abs(m_gpu[g] - r.mass) <= 1e-5 * r.mass + 1e-7, (step, g, m_gpu[g], r.mass)
            else:
                assert m_gpu[g] == -1.0
            exp_tok = -1 if r.token is None else r.token
            if t_gpu[g] != exp_tok:
                # only a continue/discard flip at the rho boundary is allowed
                assert r.soft and abs(r.mass - rho) <= 2e-5 * max(rho, r.mass), (step, g, t_gpu[g], exp_tok)
                boundary += 1
                return boundary, soft, deep  # the two runs have diverged; stop comparing this loop
            assert got["decision"][g] == ref[g].decision, (step, g)
            assert got["done"][g] == int(ref[g].done), (step, g)
            assert got["decisive_step"][g] == ref[g].decisive_step, (step, g)
            assert got["steps"][g] == ref[g].steps and got["length"][g] == len(ref[g].q), (step, g)
        ref_active = ogate.row_mask_update(ref, rpg, ref_active)
        assert np.array_equal(active.cpu().numpy(), ref_active), step
    trie.close()
    return boundary, soft, deep


@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_soft_gate_loops_small_vocab(gpu_lib, seed, dtype):
    P = workloads.make_refusal_set(12, 2, 6, 300, seed, avoid=[7])
    boundary, soft, deep = _run_loop(P, eos=7, groups=24, vocab=300, steps=8, c=5, k=20, rho=0.05, max_len=12,
                               seed=seed, dtype=dtype)
    assert soft > 0 and boundary <= 1


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_soft_gate_unaligned_rows(gpu_lib, dtype):
    # vocabulary 301: row starts off 16-byte boundaries, so the kernel reads
    # single elements instead of staging 16-byte vectors
    P = workloads.make_refusal_set(12, 2, 6, 301, 3, avoid=[7])
    boundary, soft, deep = _run_loop(P, eos=7, groups=24, vocab=301, steps=8, c=5, k=20, rho=0.05, max_len=12,
                                     seed=3, dtype=dtype)
    assert soft > 0 and boundary <= 1


def test_soft_gate_many_candidates_and_large_k(gpu_lib):
    # 600 refusal sequences: the root has hundreds of children; K = 100 needs several ranking passes
    P = workloads.make_refusal_set(600, 2, 8, 4000, 5)
    boundary, soft, deep = _run_loop(P, eos=-1, groups=16, vocab=4000, steps=5, c=3, k=100, rho=0.02, max_len=8,
                                     seed=5, boost=0.9, scale=1.0)
    assert soft > 0 and boundary <= 1
    assert deep > 0  # the sort-and-search path ran


def test_soft_gate_llama_vocab(gpu_lib):
    P = workloads.make_refusal_set(64, 2, 8, 128256, 9, avoid=[128009])
    boundary, soft, deep = _run_loop(P, eos=128009, groups=16, vocab=128256, steps=4, c=4, k=40, rho=0.1, max_len=32,
                               seed=9, boost=0.8)
    assert soft > 0 and boundary <= 1


def test_soft_gate_paper_illustration(gpu_lib):
    import torch
    V = GOLDEN_VOCAB
    P = [[V.index("I"), V.index("cannot")], [V.index("I"), V.index("can't")],
         [V.index("I"), V.index("'m"), V.index("sorry")]]
    eos = V.index("<eos>")
    probs = np.array([0.04, 0.40, 0.15, 0.10, 0.08, 0.02, 0.20, 0.01])
    for k, rho, exp_tok in ((5, 0.20, "cannot"), (5, 0.40, None), (4, 0.30, None), (2, 0.0, None),
                            (8, 0.335, "cannot")):
        trie = binding.Trie(P, 2)
        st = binding.new_gate_state(1)
        binding.rgd_gate_state_init(st, 1)
        tok = torch.empty(1, dtype=torch.int32, device="cuda")
        first = torch.full((1, 8), -10.0, dtype=torch.float32, device="cuda")
        first[0, V.index("I")] = 0.0  # the partial probe "I"
        binding.rgd_soft_gate(trie, 1, 1, first, 8, k, rho, 4, eos, 16, st, tok)
        logits = torch.from_numpy(np.log(probs).astype(np.float32)).cuda().view(1, 8)
        mass = torch.empty(1, dtype=torch.float32, device="cuda")
        binding.rgd_soft_gate(trie, 1, 1, logits, 8, k, rho, 4, eos, 16, st, tok, mass_out=mass)
        torch.cuda.synchronize()
        got = binding.decode_gate_state(st)
        if exp_tok is None:
            assert int(tok.item()) == -1 and got["decision"][0] == ogate.NON_REFUSAL and got["done"][0] == 1
        else:
            assert int(tok.item()) == V.index(exp_tok) and got["done"][0] == 0
            assert got["decision"][0] == ogate.REFUSAL  # "I cannot" is a whole two-token opening
        trie.close()
