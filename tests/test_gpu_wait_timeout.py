"""A bounded wait of the attention kernel that runs out, on purpose and safely.

The kernel's blocks never wait without a limit: a split job's merger waits for
its other pieces to count themselves in the job's counter, and gives up after
the limit (rgd_set_wait_limit_ns).  Here every counter of the caller's
workspace starts at a value no set of pieces can complete, so every merger's
wait runs out: the call must come back (within about the short limit, not the
2 s default), report RGD_DEV_WAIT_TIMEOUT in the status word, and leave the
context usable -- the same call on a fresh workspace then matches the oracle.
No GPU fault is involved: nothing traps, every wait ends by its clock."""
import time

import numpy as np
import pytest

from oracle import attention as oattn
from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


def _case():
    return workloads.make_attn_case("timeout", 3, 3, 8, 2, 128, [0, 37, 300], [0, 1, 16, 17, 40, 0, 5, 33, 64],
                                    seed=9)


def test_merger_wait_runs_out_and_reports(gpu_lib):
    import torch
    case = _case()
    J = case.num_groups * case.num_kv_heads
    dev = device.attn_to_device(case, num_ctas=7)  # 74 pages over 7 blocks: the long jobs are split
    dev.workspace[: 4 * J].view(torch.int32).fill_(0x7777)  # no count of pieces reaches this
    torch.cuda.synchronize()
    binding.rgd_set_wait_limit_ns(20_000_000)  # 20 ms
    try:
        t0 = time.perf_counter()
        dev.run()
        torch.cuda.synchronize()
        dt = time.perf_counter() - t0
    finally:
        binding.rgd_set_wait_limit_ns(0)
    status = int(dev.dev_status.item())
    assert status & binding.RGD_DEV_WAIT_TIMEOUT, status
    assert dt < 1.0, dt  # the short limit applied (the default is 2 s per wait)
    # the context is usable: the same call on a fresh workspace matches the oracle
    dev2 = device.attn_to_device(case, num_ctas=7)
    dev2.run()
    torch.cuda.synchronize()
    assert int(dev2.dev_status.item()) == 0
    o = dev2.out.float().cpu().numpy()
    ref_o, _ = oattn.decode_attention_case(case)
    assert np.all(np.abs(o - ref_o) <= ATOL + RTOL * np.abs(ref_o))
    assert np.all(dev2.workspace[: 4 * J].view(torch.int32).cpu().numpy() == 0)
