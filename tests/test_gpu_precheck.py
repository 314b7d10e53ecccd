"""The residual-stream precheck (App. A) on the GPU against the fp64 oracle.

Decisions are compared bit for bit except where the exact logit lies within
fp32 accumulation error of the threshold's logit (the kernel sums d fp32
products; the bound below is d * 2^-23 * sum |w_i h_i| plus the bias's and
the logistic's own rounding); such groups are counted, and must be rare.
Probabilities within 1e-6 absolute + 1e-5 relative.
"""
import math

import numpy as np
import pytest

from oracle import gate as ogate
from oracle import precheck as opre
from paper_2607_20791_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


def _h32(case):
    if case.dtype == "f32":
        return case.h.astype(np.float64)
    return (case.h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _run(case, pre_steps=None):
    import torch
    G, rpg = case.groups, case.rows_per_group
    if case.dtype == "f32":
        h = torch.from_numpy(case.h).cuda()
    else:
        h = torch.from_numpy(case.h.view(np.int16)).cuda().view(torch.bfloat16)
    w = torch.from_numpy(case.w).cuda()
    st = binding.new_gate_state(G)
    binding.rgd_gate_state_init(st, G)
    if pre_steps:  # mark some probes as already begun (a token consumed)
        host = st.cpu().numpy()
        for g in pre_steps:
            host[g, 8:12] = np.frombuffer(np.int32(1).tobytes(), np.uint8)
        st.copy_(torch.from_numpy(host))
    active = torch.ones(G * rpg, dtype=torch.uint8, device="cuda")
    prob = torch.full((G,), -1.0, dtype=torch.float32, device="cuda")
    binding.rgd_residual_precheck(h, w, case.b, case.theta, rpg, st, active, prob)
    torch.cuda.synchronize()
    return binding.decode_gate_state(st), active.cpu().numpy(), prob.cpu().numpy()


def _check(case, pre_steps=()):
    got, active, prob = _run(case, pre_steps)
    h = _h32(case)
    z, p, skip = opre.precheck(h, case.w, case.b, case.theta)
    states = [ogate.GateState() for _ in range(case.groups)]
    for g in pre_steps:
        states[g].steps = 1
    ref_active = opre.apply(states, skip, case.rows_per_group, np.ones(case.groups * case.rows_per_group, np.uint8))
    assert np.all(np.abs(prob - p) <= 1e-6 + 1e-5 * p), float(np.abs(prob - p).max())
    zt = math.log(case.theta / (1.0 - case.theta)) if 0.0 < case.theta < 1.0 else None
    mag = np.abs(h * case.w.astype(np.float64)).sum(axis=1) + abs(case.b)
    boundary = 0
    for g in range(case.groups):
        near = zt is not None and abs(z[g] - zt) <= case.d * 2.0 ** -23 * mag[g] + 1e-5 * (1 + abs(zt))
        same = (got["decision"][g] == states[g].decision and got["done"][g] == int(states[g].done)
                and active[g * case.rows_per_group] == ref_active[g * case.rows_per_group])
        if not same:
            assert near, (g, z[g], zt)
            boundary += 1
        assert got["decisive_step"][g] == -1 and got["node"][g] == 0
    # sample rows are never touched
    for g in range(case.groups):
        assert np.all(active[g * case.rows_per_group + 1:(g + 1) * case.rows_per_group] == 1)
    assert boundary <= max(1, case.groups // 100)
    return skip


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("G,d", [(1, 1), (3, 100), (16, 4096), (257, 3584)])
def test_precheck_matches_oracle(gpu_lib, dtype, G, d):
    case = workloads.make_precheck_case("pre", G, d, dtype, 0.5, seed=G + d, weight_scale=4.0)
    skip = _check(case)
    if G >= 16:
        assert 0 < skip.sum() < G  # both outcomes exercised


def test_precheck_llama_shaped_threshold(gpu_lib):
    case = workloads.llama8b_precheck(seed=0)
    skip = _check(case)
    assert 0 < skip.sum() < case.groups


def test_precheck_extremes_and_started_probes(gpu_lib):
    case = workloads.make_precheck_case("pre1", 20, 512, "f32", 1.0, seed=3)
    _check(case, pre_steps=[2, 5])  # theta = 1: every fresh group skips, started ones stay
    case = workloads.make_precheck_case("pre0", 20, 512, "bf16", 0.0, seed=4)
    skip = _check(case)  # theta = 0: no group skips (p > 0)
    assert not skip.any()
