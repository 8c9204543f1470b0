"""GPU parity of binary64 operands (peat_compare, peat_compare_segmented)
against the oracle: integer outputs bit-exact, max_abs / max_rel bit-identical,
sums within the stated bound (exact by design)."""
import math

import numpy as np
import pytest
import torch

from parity_util import assert_hist_equal, assert_stats_equal, f64_pairs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0, max_segments=5000)
    yield handle
    handle.close()


def dev(bits, offset=0):
    buf = torch.empty(bits.size + offset, dtype=torch.int64, device="cuda")
    buf[offset:].copy_(torch.from_numpy(bits.view(np.int64).copy()))
    return buf.view(torch.float64)[offset:]


def check(peat, oracle, h, gb, cb, rtol, atol, goff=0, coff=0, ctx=""):
    st, hist = peat.peat_compare(h, dev(gb, goff), dev(cb, coff), rtol, atol)
    ost, ohist = oracle.compare(gb, cb, "f64", rtol, atol)
    assert_stats_equal(st, ost, ctx)
    assert_hist_equal(hist, ohist, ctx)
    return st


@pytest.mark.parametrize("n", [1, 2, 3, 4095, 100_003, (1 << 20) + 3])
def test_f64_mixtures(peat_gpu, oracle, h, n):
    gb, cb = f64_pairs(n, seed=n)
    for rtol, atol in ((0.0, 0.0), (1e-9, 1e-300), (1e-3, 0.0)):
        check(peat_gpu, oracle, h, gb, cb, rtol, atol, ctx=f"n={n} tol={rtol},{atol}")


def test_f64_misaligned_and_segments(peat_gpu, oracle, h):
    n = 200_001
    gb, cb = f64_pairs(n, seed=5)
    check(peat_gpu, oracle, h, gb, cb, 1e-6, 0.0, goff=1, coff=1, ctx="both misaligned")
    check(peat_gpu, oracle, h, gb, cb, 1e-6, 0.0, goff=1, coff=0, ctx="one misaligned")
    rng = np.random.default_rng(6)
    cuts = np.sort(rng.choice(np.arange(1, n), 60, replace=False))
    off = np.concatenate([[0], cuts[:30], cuts[29:30], cuts[30:], [n, n]])
    sts, hists = peat_gpu.peat_compare_segmented(h, dev(gb), dev(cb), off.tolist(), 1e-6, 1e-300)
    osts, ohists = oracle.compare_segmented(gb, cb, off, "f64", 1e-6, 1e-300)
    for s in range(len(osts)):
        assert_stats_equal(sts[s], osts[s], f"segment {s}")
        assert_hist_equal(hists[s], ohists[s], f"segment {s}")


def test_f64_tolerance_ties(peat_gpu, oracle, h):
    """|c - g| equal to rtol |g| + atol exactly, and one binary64 step either side."""
    rng = np.random.default_rng(7)
    n = 20_000
    g = rng.standard_normal(n) * np.exp2(rng.integers(-30, 30, n))
    rtol = 2.0 ** -20
    c = g + rtol * np.abs(g)  # exact: |g| 2^-20 is a multiple of the step of g
    step = rng.integers(-1, 2, n)
    cb = (c.view(np.uint64).astype(np.int64) + step).astype(np.uint64)
    st = check(peat_gpu, oracle, h, g.view(np.uint64).copy(), cb, rtol, 0.0, ctx="ties")
    assert st["count"][1] > 0 and st["count"][2] > 0


def test_f64_range_edges(peat_gpu, oracle, h):
    big, tiny = 1.7976931348623157e308, 5e-324
    g = np.array([-big, 0.0, tiny, 2 * tiny, 1e-300, big, -0.0, np.inf, np.nan, 1.0], np.float64)
    c = np.array([big, 3 * tiny, 0.0, 0.0, 1e10, -big, 0.0, np.inf, np.nan, -np.inf], np.float64)
    check(peat_gpu, oracle, h, g.view(np.uint64).copy(), c.view(np.uint64).copy(), 0.0, 0.0, ctx="edges")
    check(peat_gpu, oracle, h, g[1:5].view(np.uint64).copy(), c[1:5].view(np.uint64).copy(), 0.0, 0.0,
          ctx="subnormal sums")


def test_fp32_candidate_against_fp64_golden(peat_gpu, oracle, h):
    """Fig. 5's FP32-FP64 pairs: a binary64 golden against its float32 rounding, widened exactly."""
    rng = np.random.default_rng(8)
    g = rng.standard_normal(1 << 20) * 3
    c = g.astype(np.float32).astype(np.float64)
    st = check(peat_gpu, oracle, h, g.view(np.uint64).copy(), c.view(np.uint64).copy(), 1e-7, 0.0, ctx="fp32 vs fp64")
    assert st["max_rel"] <= 2.0 ** -24 and st["max_ulp"] <= 1 << 28


def test_other_entry_points_refuse_f64(peat_gpu, h):
    x = torch.zeros(64, dtype=torch.float64, device="cuda")
    for call in (lambda: peat_gpu.peat_topk_mean(h, x, x), lambda: peat_gpu.peat_tensor_stats(h, x),
                 lambda: peat_gpu.peat_pseudo_error_inject(h, x, [dict(kind="bias", x=1e-3)], 1),
                 lambda: peat_gpu.peat_compare_noalloc(x, x, 1e-3)):
        with pytest.raises(peat_gpu.PeatError) as e:
            call()
        assert e.value.status == 2


@pytest.mark.parametrize("n", [1, 3, 4099, 100_003])
def test_f64_isclose_grid(peat_gpu, oracle, h, n):
    gb, cb = f64_pairs(n, seed=70 + n)
    rtols = [0.0, 1e-12, 1e-9, 1e-6, 1e-3, 1.0]
    atols = [1e-300, 0.0, 1e-12, 1e30, 1e-6]
    for goff in (0, 1):
        got = peat_gpu.peat_isclose_grid(h, dev(gb, goff), dev(cb, goff), rtols, atols)
        want = oracle.isclose_grid(gb, cb, "f64", rtols, atols)
        assert np.array_equal(got, want), (n, goff, got, want)


def test_f64_isclose_fig5_fp32_vs_fp64(peat_gpu, oracle, h):
    """Fig. 5's FP32-FP64 pass fractions: a binary64 golden against its float32 rounding."""
    rng = np.random.default_rng(12)
    g = rng.standard_normal(300_000) * np.exp2(rng.integers(-8, 8, 300_000))
    c = g.astype(np.float32).astype(np.float64)
    rtols = [0.0, 1e-9, 1e-8, 3e-8, 6e-8, 1e-7, 1e-6]
    atols = [0.0, 1e-12, 1e-9, 1e-6]
    gb, cb = g.view(np.uint64).copy(), c.view(np.uint64).copy()
    got = peat_gpu.peat_isclose_grid(h, dev(gb), dev(cb), rtols, atols)
    want = oracle.isclose_grid(gb, cb, "f64", rtols, atols)
    assert np.array_equal(got, want)
    assert got[-1, 0] == g.size and got[0, 0] < g.size  # rtol 1e-6 accepts every float32 rounding
