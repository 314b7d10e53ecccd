"""Shared-prefix split-KV decode attention on the GPU vs the fp64 oracle.

Tolerance (bf16 output): |gpu - ref| <= 2e-3 + 1e-2 * |ref| elementwise, and the
LSE within 1e-3 + 1e-4 * |ref|."""
import numpy as np
import pytest

from oracle import attention as oattn
from paper_2607_20791_gb300 import binding, device, workloads

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2


def _run(case, **kw):
    import torch
    dev = device.attn_to_device(case, **kw)
    dev.run()
    torch.cuda.synchronize()
    return dev


def _check(case, dev, rows=None, expect_status=0):
    import torch
    assert int(dev.dev_status.item()) == expect_status
    o = dev.out.float().cpu().numpy()
    lse = dev.lse.cpu().numpy()
    ref_o, ref_l = oattn.decode_attention_case(case, rows=rows)
    rows = range(case.num_rows) if rows is None else rows
    worst = 0.0
    for r in rows:
        if not case.row_active[r]:
            assert np.all(o[r] == 0) and np.all(np.isnan(lse[r])), r  # untouched
            continue
        err = np.abs(o[r] - ref_o[r])
        lim = ATOL + RTOL * np.abs(ref_o[r])
        assert np.all(err <= lim), (r, float(err.max()), float((err - lim).max()))
        worst = max(worst, float(err.max()))
        fin = np.isfinite(ref_l[r])
        assert np.array_equal(np.isfinite(lse[r]), fin), r
        assert np.allclose(lse[r][fin], ref_l[r][fin], atol=1e-3, rtol=1e-4), r
    # the split-job counters at the start of the workspace are back at zero
    J = case.num_groups * case.num_kv_heads
    tickets = dev.workspace[: 4 * J].view(torch.int32).cpu().numpy()
    assert np.all(tickets == 0), tickets
    return worst


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("ctas", [0, 1, 2, 3, 7, 29, 64, 200])
def test_small_multi_tile_ragged(gpu_lib, D, ctas):
    # 1 block (every job in one block), a few blocks (jobs split at ragged page
    # boundaries), and more blocks than pages (empty blocks, one-page pieces)
    case = workloads.make_attn_case("small", 3, 3, 8, 2, D, [0, 37, 300],
                                    [0, 1, 16, 17, 40, 0, 5, 33, 64], seed=D + ctas)
    _check(case, _run(case, num_ctas=ctas))


def test_tiny_config(gpu_lib):
    for step in range(3):
        case = workloads.tiny(seed=1, step=step).attn
        _check(case, _run(case))


def test_llama8b_full(gpu_lib):
    case = workloads.llama8b(seed=0).attn
    _check(case, _run(case))


@pytest.mark.parametrize("ctas", [13, 1000])
def test_llama8b_other_block_counts(gpu_lib, ctas):
    case = workloads.llama8b(seed=1).attn
    _check(case, _run(case, num_ctas=ctas), rows=list(range(0, 80, 7)))


def test_query_tiles_per_group(gpu_lib):
    # rows_per_group * Hq/Hkv = 1*4 (one tile), 3*8 (two query tiles), 16*8 = 128 (eight tiles)
    for rpg, Hq in [(1, 32), (3, 64), (16, 64)]:
        case = workloads.make_attn_case("q", 2, rpg, Hq, 8, 128, [100, 260], list(range(0, 2 * rpg)),
                                        seed=rpg)
        _check(case, _run(case, num_ctas=5))


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("rpg,Hq,Hkv,ctas", [(11, 24, 8, 0), (5, 64, 8, 3), (8, 64, 8, 1), (12, 64, 8, 7)])
def test_query_copy_counts(gpu_lib, D, rpg, Hq, Hkv, ctas):
    # queries per kv head 33, 40, 64 (two copies of the queries in the tensor
    # memory lanes) and 96 (one copy over three lane quarters), with jobs split
    # over blocks and whole jobs in one block
    G = 3
    slens = [(7 * i) % 70 for i in range(G * rpg)]
    case = workloads.make_attn_case("copies", G, rpg, Hq, Hkv, D, [0, 45, 230], slens, seed=rpg + D)
    _check(case, _run(case, num_ctas=ctas))


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("rpg", [1, 3, 5, 7, 8])
@pytest.mark.parametrize("ctas", [0, 7])
def test_softmax_set_counts(gpu_lib, D, rpg, ctas):
    # queries per kv head 4, 12, 20, 28 and 32: one to four sets of eight query
    # columns in the transposed kernel (the last set partly or wholly padding
    # for 4, 12, 20 and 28), jobs whole in one block and split over blocks
    G = 3
    slens = [(11 * i) % 90 for i in range(G * rpg)]
    case = workloads.make_attn_case("sets", G, rpg, 32, 8, D, [0, 45, 230], slens, seed=100 + rpg + D)
    _check(case, _run(case, num_ctas=ctas))


def test_masked_rows_and_groups(gpu_lib):
    active = np.array([1, 0, 1, 0, 0, 0, 0, 1, 1], np.uint8)  # group 1 fully masked
    case = workloads.make_attn_case("mask", 3, 3, 8, 2, 128, [50, 70, 90], [3, 4, 5, 6, 7, 8, 0, 0, 20],
                                    seed=3, row_active=active)
    _check(case, _run(case))


def test_bad_page_ids_are_flagged(gpu_lib):
    case = workloads.make_attn_case("bad", 1, 2, 4, 1, 128, [40], [8, 0], seed=2)
    case.prompt_block_table[0, 1] = case.num_pages + 5
    dev = _run(case)
    assert int(dev.dev_status.item()) & binding.RGD_DEV_BAD_PAGE
    # the out-of-range page reads as zeros: equals attention with that page zeroed
    fixed = workloads.make_attn_case("bad", 1, 2, 4, 1, 128, [40], [8, 0], seed=2)
    page = int(fixed.prompt_block_table[0, 1])
    fixed.k_pages[page] = 0
    fixed.v_pages[page] = 0
    o = dev.out.float().cpu().numpy()
    ref_o, _ = oattn.decode_attention_case(fixed)
    assert np.all(np.abs(o - ref_o) <= ATOL + RTOL * np.abs(ref_o))


def test_repeated_calls_reuse_workspace(gpu_lib):
    import torch
    case = workloads.make_attn_case("rep", 2, 5, 32, 8, 128, [513, 1000], list(range(0, 200, 20)), seed=6)
    dev = device.attn_to_device(case)
    for _ in range(3):
        dev.out.zero_()
        dev.run()
    torch.cuda.synchronize()
    _check(case, dev)
