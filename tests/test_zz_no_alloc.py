"""The allocation-free attention entry point against the workspace one.

rgd_prefix_decode_attn_noalloc serves callers that cannot allocate device memory
(for instance inside a serving engine whose KV-cache manager has reserved the free
memory, or on a decode loop where cudaMalloc would synchronise the device): it
uses a fixed scratch array inside the library instead of a caller workspace.
Two calls in a row, on different shapes, through the C ABI, must match the
workspace entry point within the attention tolerance used everywhere else.
This file is collected last on purpose."""
import numpy as np
import pytest

from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


def _both(case):
    import torch
    ref = device.attn_to_device(case)
    ref.run()
    out = torch.zeros_like(ref.out)
    lse = torch.full_like(ref.lse, float("nan"))
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    binding.rgd_prefix_decode_attn_noalloc(ref.shape, ref.q, ref.k_pages, ref.v_pages, ref.prompt_block_table,
                                           ref.prompt_len, ref.suffix_block_table, ref.suffix_len,
                                           ref.row_active, ref.softmax_scale, out, lse, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0 and int(ref.dev_status.item()) == 0
    a, b = out.float().cpu().numpy(), ref.out.float().cpu().numpy()
    assert np.all(np.abs(a - b) <= ATOL + RTOL * np.abs(b))
    la, lb = lse.cpu().numpy(), ref.lse.cpu().numpy()
    fin = np.isfinite(lb)
    assert np.array_equal(np.isfinite(la), fin)
    assert np.allclose(la[fin], lb[fin], atol=1e-3, rtol=1e-4)


def test_noalloc_matches_workspace_entry_point_twice(gpu_lib):
    # first call: the Llama-3-8B-shaped step; second call: a smaller shape with
    # masked rows, which must not see the first call's partials
    _both(workloads.llama8b(seed=2).attn)
    active = np.array([1, 0, 1, 1, 1, 1, 0, 0, 1], np.uint8)
    _both(workloads.make_attn_case("second", 3, 3, 8, 2, 64, [0, 37, 300], [0, 1, 16, 17, 40, 0, 5, 33, 64],
                                   seed=5, row_active=active))


def test_noalloc_rejects_oversized_shapes(gpu_lib):
    import torch
    case = workloads.high_batch(seed=0, with_kv=False).attn  # 2048 (group, kv head) jobs
    shape = device.attn_shape(case, num_ctas=152)
    assert binding.rgd_prefix_decode_attn_workspace_size(shape) > (8 << 20)
    t = torch.zeros(16, dtype=torch.int32, device="cuda")
    b = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    # raw pointers: the binding passes them through unchecked, so this reaches
    # the library's own workspace check, which comes before any launch
    tp, bp = t.data_ptr(), b.data_ptr()
    with pytest.raises(binding.RgdError) as ei:
        binding.rgd_prefix_decode_attn_noalloc(shape, bp, bp, bp, tp, tp, tp, tp, None, 0.1, bp, None)
    assert ei.value.code == binding.RGD_ERR_UNSUPPORTED
