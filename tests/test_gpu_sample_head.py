"""Sample head on the GPU vs the oracle: probe tokens and min-p sets bit-exact,
sampled tokens bit-exact except where the oracle flags the uniform draw as
within 1e-6 of a CDF boundary (those are counted)."""
import numpy as np
import pytest

from oracle import sampling as osamp
from paper_2607_20791_gb300 import device, workloads

pytestmark = pytest.mark.gpu


def _run(case, with_mask=True):
    import torch
    dev = device.head_to_device(case, with_mask=with_mask)
    dev.run(with_mask=with_mask)
    torch.cuda.synchronize()
    return dev


def _check(case, dev, rows=None, check_mask=True):
    tok = dev.token_out.cpu().numpy()
    cnt = dev.kept_count.cpu().numpy()
    mask = dev.kept_mask.cpu().numpy() if (check_mask and dev.kept_mask is not None) else None
    assert int(dev.dev_status.item()) == 0
    ref = osamp.sample_head(case.logits, case.dtype, case.is_probe, case.temperature, case.min_p,
                            case.seed, case.step, case.row_active, rows=rows)
    rows = range(case.rows) if rows is None else rows
    boundary_mismatch = 0
    for r in rows:
        if not case.row_active[r]:
            assert tok[r] == -1 and cnt[r] == 0, r
            continue
        greedy = bool(case.is_probe[r]) or float(case.temperature[r]) == 0.0
        if greedy:
            assert tok[r] == ref.tokens[r], (r, tok[r], ref.tokens[r])
            assert cnt[r] == 1
            continue
        assert cnt[r] == ref.kept_count[r], (r, cnt[r], ref.kept_count[r])
        if mask is not None:
            assert np.array_equal(mask[r].astype(bool), ref.kept[r]), r
        if tok[r] != ref.tokens[r]:
            assert ref.boundary[r], (r, tok[r], ref.tokens[r])
            assert ref.kept[r][tok[r]]
            boundary_mismatch += 1
    return boundary_mismatch


def test_tiny_head(gpu_lib):
    for step in range(4):
        case = workloads.tiny(seed=step, step=step).head
        assert _check(case, _run(case)) == 0


def test_llama8b_head_full(gpu_lib):
    case = workloads.llama8b(seed=0, with_kv=False).head
    assert _check(case, _run(case)) == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("vocab", workloads.SWEEP_VOCABS)
@pytest.mark.parametrize("batch", [1, 8, 64])
def test_sweep_small_batches(gpu_lib, batch, vocab, dtype):
    case = workloads.head_sweep(batch, vocab, dtype, seed=batch + vocab)
    assert _check(case, _run(case)) == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("batch", [128, 300, 500])
def test_several_waves(gpu_lib, batch, dtype):
    # 128, 300 and 500 rows at 8 CTAs per row are more CTAs than the device
    # holds at once (5 per SM): clusters run in several waves; every row and
    # kept mask compared
    case = workloads.head_sweep(batch, 32000, dtype, seed=7 + batch)
    assert _check(case, _run(case)) == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("vocab", [1, 7, 33, 1000, 4097, 32001])
def test_ragged_vocab(gpu_lib, vocab, dtype):
    # rows start at unaligned addresses; slices end in ragged tails; tiny vocabularies
    rng = np.random.default_rng(vocab)
    l = (2.0 * rng.standard_normal((9, vocab))).astype(np.float32)
    case = workloads.make_head_case("ragged", l, dtype, [1, 0, 0, 0, 0, 0, 0, 0, 0],
                                    [0, 1.0, 2.0, 0.5, 3.0, 10.0, 1.0, 1e-4, 0.0],
                                    [0, 0.1, 0.0, 0.3, 0.05, 0.0, 1.0, 0.0, 0.2], seed=vocab)
    assert _check(case, _run(case)) == 0


def test_exact_ties_lowest_index(gpu_lib):
    V = 50000
    l = np.full((6, V), -3.0, np.float32)
    l[0, [17, 4000, 49999]] = 5.0          # ties in different CTA slices
    l[1, [6250, 6251]] = 2.0               # ties across a slice boundary
    l[2, :] = 0.0                          # all equal
    l[3, [49999]] = 1.0
    l[4, [0, 49999]] = 1.0
    l[5, [31250, 12]] = 9.0
    case = workloads.make_head_case("ties", l, "f32", [1] * 6, [0.0] * 6, [0.0] * 6, seed=1)
    dev = _run(case)
    assert dev.token_out.cpu().numpy().tolist() == [17, 6250, 0, 49999, 0, 12]
    case_b = workloads.make_head_case("ties", l, "bf16", [0] * 6, [0.0] * 6, [0.0] * 6, seed=1)
    assert _check(case_b, _run(case_b)) == 0


def test_min_p_one_and_temperature_limits(gpu_lib):
    l = workloads.zipf_logits(6, 32000, seed=4)
    case = workloads.make_head_case("lim", l, "f32", [0] * 6, [1.0, 1e-4, 10.0, 2.0, 5.0, 0.5],
                                    [1.0, 0.0, 0.0, 1.0, 0.3, 0.05], seed=4)
    dev = _run(case)
    tok = dev.token_out.cpu().numpy()
    assert tok[0] == np.argmax(l[0]) and tok[1] == np.argmax(l[1]) and tok[3] == np.argmax(l[3])
    assert dev.kept_count.cpu().numpy()[2] == 32000
    assert _check(case, dev) == 0


def test_inactive_rows_and_bad_params(gpu_lib):
    import torch
    l = workloads.zipf_logits(5, 4096, seed=8)
    case = workloads.make_head_case("inact", l, "f32", [1, 0, 0, 0, 0], [0, 1.0, 1.0, -1.0, 1.0],
                                    [0, 0.1, 0.1, 0.1, 2.0], seed=8, row_active=[1, 0, 1, 1, 1])
    dev = _run(case)
    tok = dev.token_out.cpu().numpy()
    assert tok[1] == -1 and tok[3] == -1 and tok[4] == -1
    assert int(dev.dev_status.item()) & 8
    ref = osamp.sample_head(case.logits, "f32", case.is_probe, case.temperature, case.min_p,
                            case.seed, 0, case.row_active, rows=[0, 2])
    assert tok[0] == ref.tokens[0]
    assert tok[2] == ref.tokens[2] or ref.boundary[2]


def test_steps_change_the_draw(gpu_lib):
    l = np.zeros((1, 1024), np.float32)  # uniform: the draw is u * 1024
    toks = []
    for step in range(8):
        case = workloads.make_head_case("u", l, "f32", [0], [1.0], [0.0], seed=5, step=step)
        dev = _run(case)
        ref = osamp.sample_row(l[0], False, 1.0, 0.0, int(case.seed[0]), step)
        assert dev.token_out.item() == ref.token or ref.boundary
        toks.append(dev.token_out.item())
    assert len(set(toks)) > 4
