"""The allocation-free attention entry point against the workspace one.

rgd_prefix_decode_attn_noalloc serves callers that cannot allocate device memory
(for instance inside a serving engine whose KV-cache manager has reserved the free
memory, or on a decode loop where cudaMalloc would synchronise the device): it
uses a fixed scratch array inside the library instead of a caller workspace.
It runs the same kernel with the same shape and block count as
rgd_prefix_decode_attn, so its outputs must be bit-identical to that entry
point's, call after call, whatever the earlier calls' shapes left in the shared
array: a small shape whose jobs are split over blocks (it writes partials),
then a shape with many more jobs (its counters must not meet those partials),
then the small one again.  The small case is also checked against the oracle.
This file is collected last on purpose."""
import numpy as np
import pytest

from oracle import attention as oattn
from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


def _both(case, num_ctas=0):
    """Runs both entry points on `case`; returns the allocation-free outputs."""
    import torch
    ref = device.attn_to_device(case, num_ctas=num_ctas)
    ref.run()
    out = torch.zeros_like(ref.out)
    lse = torch.full_like(ref.lse, float("nan"))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    binding.rgd_prefix_decode_attn_noalloc(ref.shape, ref.q, ref.k_pages, ref.v_pages, ref.prompt_block_table,
                                           ref.prompt_len, ref.suffix_block_table, ref.suffix_len,
                                           ref.row_active, ref.softmax_scale, out, lse, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0 and int(ref.dev_status.item()) == 0
    assert torch.equal(out.view(torch.int16), ref.out.view(torch.int16))
    assert torch.equal(lse.view(torch.int32), ref.lse.view(torch.int32))
    return out.float().cpu().numpy(), lse.cpu().numpy()


def _small():
    active = np.array([1, 0, 1, 1, 1, 1, 0, 0, 1], np.uint8)
    return workloads.make_attn_case("second", 3, 3, 8, 2, 64, [0, 37, 300], [0, 1, 16, 17, 40, 0, 5, 33, 64],
                                    seed=5, row_active=active)


def test_noalloc_matches_workspace_entry_point_across_shapes(gpu_lib):
    small = _small()
    # 7 blocks over the small case's 6 jobs: every job with pages is split
    for case, ctas in ((small, 7), (workloads.llama8b(seed=2).attn, 0), (small, 7)):
        o, lse = _both(case, ctas)
        if case is small:
            ref_o, ref_l = oattn.decode_attention_case(small)
            on = small.row_active.astype(bool)
            assert np.all(np.abs(o[on] - ref_o[on]) <= ATOL + RTOL * np.abs(ref_o[on]))
            fin = np.isfinite(ref_l[on])
            assert np.array_equal(np.isfinite(lse[on]), fin)
            assert np.allclose(lse[on][fin], ref_l[on][fin], atol=1e-3, rtol=1e-4)


def test_noalloc_rejects_oversized_shapes(gpu_lib):
    import torch
    case = workloads.high_batch(seed=0, with_kv=False).attn  # 2048 (group, kv head) jobs
    shape = device.attn_shape(case, num_ctas=152)
    assert binding.rgd_prefix_decode_attn_workspace_size(shape) > (8 << 20)
    t = torch.zeros(16, dtype=torch.int32, device="cuda")
    b = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    # raw pointers: the binding passes them through unchecked, so this reaches
    # the library's own size checks, which come before any launch
    tp, bp = t.data_ptr(), b.data_ptr()
    with pytest.raises(binding.RgdError) as ei:
        binding.rgd_prefix_decode_attn_noalloc(shape, bp, bp, bp, tp, tp, tp, tp, None, 0.1, bp, None)
    assert ei.value.code == binding.RGD_ERR_UNSUPPORTED
    # more (group, kv head) jobs than the fixed counter area holds
    big = binding.AttnShape(num_groups=8193, rows_per_group=1, num_q_heads=1, num_kv_heads=1, head_dim=64,
                            page_size=16, num_pages=16, max_prompt_pages=1, max_suffix_pages=1, num_ctas=1,
                            reserved=0)
    with pytest.raises(binding.RgdError) as ei:
        binding.rgd_prefix_decode_attn_noalloc(big, bp, bp, bp, tp, tp, tp, tp, None, 0.1, bp, None)
    assert ei.value.code == binding.RGD_ERR_UNSUPPORTED
