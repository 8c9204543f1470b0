"""GPU parity of the isclose pass counts over a tolerance grid (Section III-A,
Fig. 5): peat_isclose_grid against oracle.isclose_grid (the oracle's compare
run once per cell), and against the GPU compare run once per cell.  Counts
are exact on both sides: bit-exact equality."""
import numpy as np
import pytest
import torch

from parity_util import NP_BITS, noise_pairs, random_pairs, to_device

pytestmark = pytest.mark.gpu

DTYPES = ["f32", "f16", "bf16"]
RTOLS = [0.0, 1e-5, 1e-4, 1e-3, 2.0 ** -7, 1e-2, 0.1, 1.0]
ATOLS = [0.0, 1e-8, 1e-6, 1e-4, 1e-2, 1.0, 1e3, 1e30]


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0)
    yield handle
    handle.close()


def check(peat, oracle, h, gb, cb, dtype, rtols=RTOLS, atols=ATOLS, goff=0, coff=0, ctx=""):
    g, c = to_device(gb, dtype, goff), to_device(cb, dtype, coff)
    got = peat.peat_isclose_grid(h, g, c, rtols, atols)
    want = oracle.isclose_grid(gb, cb, dtype, rtols, atols)
    assert np.array_equal(got, want), f"{ctx}: gpu\n{got}\noracle\n{want}"
    return got


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [0, 1, 7, 4099, 100_003])
def test_random_mixtures(peat_gpu, oracle, h, dtype, n):
    gb, cb = random_pairs(dtype, n, seed=900 + n)
    check(peat_gpu, oracle, h, gb, cb, dtype, ctx=f"n={n}")


@pytest.mark.parametrize("shape", [(1, 1), (3, 5), (64, 1), (1, 64), (5, 12)])
def test_grid_shapes(peat_gpu, oracle, h, shape):
    nr, na = shape
    rtols = sorted(np.random.default_rng(nr).uniform(0, 0.05, nr).tolist())
    atols = np.random.default_rng(na).uniform(0, 1e-3, na).tolist()
    gb, cb = noise_pairs("bf16", 60_001, seed=4, rel=1e-2)
    check(peat_gpu, oracle, h, gb, cb, "bf16", rtols, atols, ctx=f"shape {shape}")


@pytest.mark.parametrize("dtype", DTYPES)
def test_misaligned_and_noise(peat_gpu, oracle, h, dtype):
    gb, cb = noise_pairs(dtype, 70_001, seed=21, rel=3e-3)
    check(peat_gpu, oracle, h, gb, cb, dtype, goff=1, coff=1, ctx="misaligned")
    check(peat_gpu, oracle, h, gb, cb, dtype, goff=3, coff=0, ctx="unequal offsets")


def test_exact_ties_float32(peat_gpu, oracle, h):
    """|c - g| equal to the float32 rounding of rtol |g| (and one step either
    side) for every rtol of the grid, with atol 0 and small atols."""
    rng = np.random.default_rng(62)
    n = 40_000
    mag = (rng.standard_normal(n) * np.exp2(rng.integers(-20, 20, n))).astype(np.float32)
    g = (mag.view(np.uint32) & np.uint32(0xFFFFF000)).view(np.float32)
    rt = [2.0 ** -7, 1e-3, 2.0 ** -3]
    parts_g, parts_c = [], []
    for r in rt:
        a = (np.abs(g).astype(np.float64) * np.float64(np.float32(r))).astype(np.float32)
        c0 = (g + a).astype(np.float32)
        for c in (c0, np.nextafter(c0, np.float32(np.inf)), np.nextafter(c0, np.float32(-np.inf))):
            parts_g.append(g)
            parts_c.append(c)
    gb = np.concatenate(parts_g).view(np.uint32)
    cb = np.concatenate(parts_c).view(np.uint32)
    check(peat_gpu, oracle, h, gb, cb, "f32", sorted(rt), [0.0, 1e-30, 1e-7], ctx="ties")


def test_agrees_with_the_compare(peat_gpu, h):
    """Every cell equals EXACT + WITHIN_TOL of peat_compare at that tolerance."""
    gb, cb = noise_pairs("f16", 500_003, seed=8, rel=2e-3)
    g, c = to_device(gb, "f16"), to_device(cb, "f16")
    rt, at = [0.0, 1e-4, 1e-3, 3e-3], [0.0, 1e-5, 1e-3]
    grid = peat_gpu.peat_isclose_grid(h, g, c, rt, at)
    for i, r in enumerate(rt):
        for j, a in enumerate(at):
            st, _ = peat_gpu.peat_compare(h, g, c, r, a)
            assert grid[i, j] == st["exact"] + st["within_tol"], (r, a)


def test_fig5_like_precision_pairs(peat_gpu, oracle, h):
    """The Fig. 5 setting: an fp32 result against the same values after an
    FP16 round trip (candidate = RN16(g) as fp32), over an rtol x atol grid."""
    rng = np.random.default_rng(5)
    g = rng.standard_normal(300_001).astype(np.float32)
    c = g.astype(np.float16).astype(np.float32)
    gb, cb = g.view(np.uint32), c.view(np.uint32)
    grid = check(peat_gpu, oracle, h, gb, cb, "f32", [1e-5, 1e-4, 1e-3, 1e-2], [0.0, 1e-8, 1e-5], ctx="fig5")
    assert grid[-1, 0] == g.size  # rtol 1e-2 accepts every FP16 rounding (relative error <= 2^-11)


def test_invalid_arguments(peat_gpu, h):
    g = torch.zeros(16, device="cuda")
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_isclose_grid(h, g, g, [1e-3, 1e-4], [0.0])      # rtols descending
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_isclose_grid(h, g, g, [0.1] * 9, [0.0] * 8)      # 72 cells
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_isclose_grid(h, g, g, [float("nan")], [0.0])


@pytest.mark.parametrize("dtype", DTYPES)
def test_repeated_and_descending_tolerances(peat_gpu, oracle, h, dtype):
    """Repeated rtols, repeated atols and atols in descending order: the kernel
    walks the atols sorted, the counts come back in the caller's order."""
    gb, cb = noise_pairs(dtype, 50_003, seed=33, rel=2e-3)
    check(peat_gpu, oracle, h, gb, cb, dtype, [0.0, 0.0, 1e-3, 1e-3, 1e-2], [1e-2, 0.0, 1e-4, 1e-2, 0.0, 1e30],
          ctx="repeated")
    check(peat_gpu, oracle, h, gb, cb, dtype, RTOLS, ATOLS[::-1], ctx="descending atols")


def test_half_the_pairs_differ(peat_gpu, oracle, h):
    """bf16 round-to-nearest against round-toward-zero of the same float32
    values (about half the pairs differ by one ulp): many full queue batches,
    vector rounds with and without an all-equal warp slot, a ragged tail."""
    n = (1 << 20) + 7
    x = torch.from_numpy(np.random.default_rng(8).standard_normal(n).astype(np.float32) * 2)
    gb = x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16).copy()
    cb = (x.view(torch.int32).numpy().view(np.uint32) >> 16).astype(np.uint16)
    got = check(peat_gpu, oracle, h, gb, cb, "bf16", ctx="rne vs rtz")
    assert got[0, 0] < n * 0.6 and got[-1, -1] == n
