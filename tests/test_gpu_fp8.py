"""GPU parity of the 8-bit formats (OCP FP8 E4M3 and E5M2): the compare,
segmented compare and isclose grid against the oracle, bit-exact counts,
histograms, indices and maxima, sums within the stated bound (exact by
design); and the entry points that do not take them say so."""
import numpy as np
import pytest
import torch

from parity_util import assert_hist_equal, assert_stats_equal

pytestmark = pytest.mark.gpu

FP8 = {"f8e4m3": torch.float8_e4m3fn, "f8e5m2": torch.float8_e5m2}


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0, max_segments=70000)
    yield handle
    handle.close()


def dev(bits, dtype, offset=0):
    buf = torch.empty(bits.size + offset, dtype=torch.uint8, device="cuda")
    buf[offset:].copy_(torch.from_numpy(bits))
    return buf.view(FP8[dtype])[offset:]


def fp8_pairs(dtype, n, seed, rel=0.05):
    """Mixture: close pairs from relative noise (float32 values rounded to the
    format), arbitrary patterns, sign flips, zeros, equal values."""
    rng = np.random.default_rng(seed)
    x = torch.from_numpy((rng.standard_normal(n) * np.exp2(rng.integers(-8, 6, n))).astype(np.float32))
    y = x * (1 + rel * torch.from_numpy(rng.standard_normal(n).astype(np.float32)))
    g = x.to(FP8[dtype]).view(torch.uint8).numpy().copy()
    c = y.to(FP8[dtype]).view(torch.uint8).numpy().copy()
    kind = rng.integers(0, 10, n)
    c = np.where(kind == 0, rng.integers(0, 256, n).astype(np.uint8), c)
    c = np.where(kind == 1, g ^ np.uint8(0x80), c)
    c = np.where(kind == 2, np.uint8(0), c)
    g = np.where(kind == 3, rng.integers(0, 256, n).astype(np.uint8), g)
    c = np.where(kind == 4, g, c)
    return g.astype(np.uint8), c.astype(np.uint8)


@pytest.mark.parametrize("dtype", list(FP8))
@pytest.mark.parametrize("n", [1, 15, 16, 17, 4095, 100_003, (1 << 20) + 9])
def test_compare_fp8(peat_gpu, oracle, h, dtype, n):
    gb, cb = fp8_pairs(dtype, n, seed=n)
    for rtol, atol in ((0.0, 0.0), (0.125, 2.0 ** -7), (1e-3, 1e-30)):
        st, hist = peat_gpu.peat_compare(h, dev(gb, dtype), dev(cb, dtype), rtol, atol)
        ost, ohist = oracle.compare(gb, cb, dtype, rtol, atol)
        assert_stats_equal(st, ost, f"{dtype} n={n} tol={rtol},{atol}")
        assert_hist_equal(hist, ohist, f"{dtype} n={n}")


@pytest.mark.parametrize("dtype", list(FP8))
def test_every_pair_of_the_type(peat_gpu, oracle, h, dtype):
    """All 65,536 pairs, each its own segment, plus the whole as one tensor."""
    g = np.repeat(np.arange(256, dtype=np.uint8), 256)
    c = np.tile(np.arange(256, dtype=np.uint8), 256)
    off = np.arange(g.size + 1)
    sts, hists = peat_gpu.peat_compare_segmented(h, dev(g, dtype), dev(c, dtype), off.tolist(), 0.125, 2.0 ** -7)
    osts, ohists = oracle.compare_segmented(g, c, off, dtype, 0.125, 2.0 ** -7)
    for s in range(g.size):
        assert_stats_equal(sts[s], osts[s], f"{dtype} pair {s:#06x}")
        assert_hist_equal(hists[s], ohists[s], f"{dtype} pair {s:#06x}")
    st, hist = peat_gpu.peat_compare(h, dev(g, dtype), dev(c, dtype), 0.125, 2.0 ** -7)
    ost, ohist = oracle.compare(g, c, dtype, 0.125, 2.0 ** -7)
    assert_stats_equal(st, ost, f"{dtype} whole")
    assert_hist_equal(hist, ohist, f"{dtype} whole")


@pytest.mark.parametrize("dtype", list(FP8))
def test_segments_misaligned_and_empty(peat_gpu, oracle, h, dtype):
    n = 300_001
    gb, cb = fp8_pairs(dtype, n, seed=7)
    rng = np.random.default_rng(5)
    cuts = np.sort(rng.choice(np.arange(1, n), 40, replace=False))
    off = np.concatenate([[0], cuts[:10], cuts[9:10], cuts[10:], [n, n]])  # one empty segment, one at the end
    for goff, coff in ((0, 0), (3, 3), (1, 6)):
        sts, hists = peat_gpu.peat_compare_segmented(h, dev(gb, dtype, goff), dev(cb, dtype, coff), off.tolist(),
                                                     1e-2, 0.0)
        osts, ohists = oracle.compare_segmented(gb, cb, off, dtype, 1e-2, 0.0)
        assert len(sts) == len(osts)
        for s in range(len(osts)):
            assert_stats_equal(sts[s], osts[s], f"{dtype} offsets {goff},{coff} seg {s}")
            assert_hist_equal(hists[s], ohists[s], f"{dtype} seg {s}")


@pytest.mark.parametrize("dtype", list(FP8))
def test_isclose_grid_fp8(peat_gpu, oracle, h, dtype):
    gb, cb = fp8_pairs(dtype, 50_001, seed=11)
    rtols = [0.0, 1e-3, 1 / 16, 0.125, 0.25, 1.0]
    atols = [1.0, 0.0, 2.0 ** -9, 2.0 ** -16, 1e-3, 100.0]
    got = peat_gpu.peat_isclose_grid(h, dev(gb, dtype), dev(cb, dtype), rtols, atols)
    want = oracle.isclose_grid(gb, cb, dtype, rtols, atols)
    assert np.array_equal(got, want), (got, want)


def test_other_entry_points_refuse_fp8(peat_gpu, h):
    g = torch.zeros(64, dtype=torch.uint8, device="cuda").view(torch.float8_e4m3fn)
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_topk_mean(h, g, g)
    assert e.value.status == 2
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_tensor_stats(h, g)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_pseudo_error_inject(h, g, [dict(kind="bias", x=1e-3)], 1)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_inject_compare(h, g, [dict(kind="bias", x=1e-3)], 1, 1e-3)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_compare_noalloc(g, g, 1e-3)


@pytest.mark.parametrize("dtype", list(FP8))
def test_mostly_equal(peat_gpu, oracle, h, dtype):
    """Long runs of bitwise-equal pairs (whole warp slots of equal 16-byte
    groups), with NaN and infinity patterns inside some equal runs and a few
    differing pairs, at aligned and misaligned bases."""
    n = (1 << 20) + 37
    rng = np.random.default_rng(41)
    gb = rng.integers(0, 256, n).astype(np.uint8)
    gb[(gb & 0x7F) == 0x7F] = 0x10  # a few NaN codes only where planted below
    cb = gb.copy()
    idx = rng.choice(n, 300, replace=False)
    cb[idx] = rng.integers(0, 256, 300).astype(np.uint8)
    gb[rng.choice(n, 20, replace=False)] = 0x7F  # NaN (both formats)
    cb[gb == 0x7F] = 0x7F
    if dtype == "f8e5m2":
        inf_at = rng.choice(n, 20, replace=False)
        gb[inf_at] = 0x7C
        cb[inf_at] = 0x7C
    for goff in (0, 5):
        st, hist = peat_gpu.peat_compare(h, dev(gb, dtype, goff), dev(cb, dtype, goff), 1e-2, 0.0)
        ost, ohist = oracle.compare(gb, cb, dtype, 1e-2, 0.0)
        assert_stats_equal(st, ost, f"{dtype} goff={goff}")
        assert_hist_equal(hist, ohist, f"{dtype} goff={goff}")
