"""GPU parity of the context statistics (Section IV-C-2): peat_tensor_stats
through the C ABI against oracle.tensor_stats.  Bar: counts exact; sum,
sum_sq, mean, var, min and max bit-identical (each the exact value rounded
once on both sides)."""
import math

import numpy as np
import pytest
import torch

from parity_util import NP_BITS, noise_pairs, random_pairs, to_device

pytestmark = pytest.mark.gpu

DTYPES = ["f32", "f16", "bf16"]
KEYS = ("n", "n_finite", "n_nan", "n_inf", "sum", "sum_sq", "mean", "var", "min", "max")


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0, max_segments=5000)
    yield handle
    handle.close()


def same(a, b):
    if isinstance(b, float):
        return a == b and math.copysign(1.0, a) == math.copysign(1.0, b)
    return a == b


def check_one(got, want, ctx):
    for k in KEYS:
        assert same(got[k], want[k]), f"{ctx}: {k} gpu={got[k]!r} oracle={want[k]!r}"


def check(peat, oracle, h, bits, dtype, offsets=None, off=0, ctx=""):
    x = to_device(bits, dtype, off)
    if offsets is None:
        check_one(peat.peat_tensor_stats(h, x), oracle.tensor_stats(bits, dtype), ctx)
        return
    got = peat.peat_tensor_stats(h, x, offsets)
    want = oracle.tensor_stats_segmented(bits, offsets, dtype)
    assert len(got) == len(want)
    for s, (a, b) in enumerate(zip(got, want)):
        check_one(a, b, f"{ctx} seg {s}")


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [0, 1, 7, 4099, 100_003])
def test_random_patterns(peat_gpu, oracle, h, dtype, n):
    g, c = random_pairs(dtype, n, seed=500 + n)
    check(peat_gpu, oracle, h, g, dtype, ctx=f"golden n={n}")
    check(peat_gpu, oracle, h, c, dtype, ctx=f"candidate n={n}")


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("off", [1, 3])
def test_misaligned(peat_gpu, oracle, h, dtype, off):
    g, _ = noise_pairs(dtype, 70_001, seed=off)
    check(peat_gpu, oracle, h, g, dtype, off=off, ctx=f"offset {off}")


@pytest.mark.parametrize("dtype", DTYPES)
def test_segments_with_empty_ones(peat_gpu, oracle, h, dtype):
    rng = np.random.default_rng(17)
    sizes = rng.integers(0, 3000, 400)
    sizes[::7] = 0
    sizes[5] = 200_000
    off = np.concatenate([[0], np.cumsum(sizes)])
    g, _ = random_pairs(dtype, int(off[-1]), seed=3)
    check(peat_gpu, oracle, h, g, dtype, offsets=off, ctx="segments")


def test_special_tensors(peat_gpu, oracle, h):
    specials = {
        "all NaN": np.full(5000, 0x7FC00000, np.uint32),
        "all zero both signs": np.array([0, 0x80000000] * 3000, np.uint32),
        "constant": np.full(100_000, np.float32(0.1).view(np.uint32), np.uint32),
        "extremes": np.array([0x7F7FFFFF, 0xFF7FFFFF, 0x00000001, 0x80000001, 0x7F800000, 0x3F800000] * 1000,
                             np.uint32),
        "wide range": (np.float32(2.0) ** np.arange(-149, 128, dtype=np.float32)).view(np.uint32),
    }
    for name, bits in specials.items():
        check(peat_gpu, oracle, h, bits, "f32", ctx=name)


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_special_16bit_tensors(peat_gpu, oracle, h, dtype):
    """The 16-bit histogram path at its edges: NaN and infinities, signed
    zeros (-0 below +0 for min and max), a constant, the largest finite and
    the smallest subnormal values, every exponent once, all bit patterns,
    and zeros next to tiny values (the window is placed by the largest
    exponent: everything far below takes the exact digit path)."""
    rng = np.random.default_rng(41)
    inf, nan, mx, sub = ((0x7C00, 0x7E00, 0x7BFF, 0x0001) if dtype == "f16" else (0x7F80, 0x7FC0, 0x7F7F, 0x0001))
    exps = 31 if dtype == "f16" else 255
    mb = 10 if dtype == "f16" else 7
    specials = {
        "all NaN": np.full(5000, nan, np.uint16),
        "all zero both signs": np.array([0, 0x8000] * 3000, np.uint16),
        "only negative zero": np.full(700, 0x8000, np.uint16),
        "constant": np.full(100_000, 0x3C00 if dtype == "f16" else 0x3F80, np.uint16),
        "extremes": np.array([mx, 0x8000 | mx, sub, 0x8000 | sub, inf, 0x8000 | inf, nan, 0] * 1000, np.uint16),
        "every exponent": np.array([(e << mb) | 3 for e in range(1, exps)] * 40
                                   + [0x8000 | (e << mb) | 5 for e in range(1, exps)] * 40, np.uint16),
        "every pattern": np.arange(65536, dtype=np.uint32).astype(np.uint16),
        "zeros and tiny": np.concatenate([np.full(3000, 0x8000, np.uint16),
                                          rng.integers(1, 1 << mb, 3000).astype(np.uint16),
                                          np.full(10, mx, np.uint16)]),
    }
    for name, bits in specials.items():
        check(peat_gpu, oracle, h, bits, dtype, ctx=name)
        perm = rng.permutation(bits.size)
        check(peat_gpu, oracle, h, bits[perm], dtype, ctx=name + " shuffled")
        check(peat_gpu, oracle, h, bits, dtype, offsets=[0, bits.size // 3, bits.size // 3, bits.size], ctx=name + " segs")


@pytest.mark.parametrize("dtype", DTYPES)
def test_scale_changes_inside_a_warp_range(peat_gpu, oracle, h, dtype):
    """Blocks of very different magnitude in one tensor: warps move their
    integer windows, and small values below a window take the digit path."""
    rng = np.random.default_rng(23)
    parts = []
    for e in [0, 20, -20, 8, -3, 30, -30]:
        e = max(min(e, 14), -14) if dtype == "f16" else e
        parts.append((rng.standard_normal(9000) * 2.0 ** e).astype(np.float32))
    x = torch.from_numpy(np.concatenate(parts))
    tdt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[dtype]
    iv = torch.int32 if dtype == "f32" else torch.int16
    bits = x.to(tdt).view(iv).numpy().view(NP_BITS[dtype])
    check(peat_gpu, oracle, h, bits, dtype, ctx="scales")


def test_repeated_calls_agree(peat_gpu, h):
    g, _ = random_pairs("bf16", 300_001, seed=8)
    x = to_device(g, "bf16")
    assert peat_gpu.peat_tensor_stats(h, x) == peat_gpu.peat_tensor_stats(h, x)


def test_workload_c3_segments(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c3_resnet50(device="cuda")
    bits = w.golden.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)
    check(peat_gpu, oracle, h, bits, "f32", offsets=w.offsets, ctx="c3 goldens")


def test_workload_c4_checkpoint_sample(peat_gpu, oracle, h):
    """The fp16 GPT-2-medium checkpoint (Laplace values over about 20 binades):
    its first 8 M elements with the workload's own segment boundaries."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c4_gpt2_medium(device="cuda")
    P = 8_000_000
    offsets = [int(o) for o in w.offsets if int(o) < P] + [P]
    bits = w.golden[:P].cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    del w
    check(peat_gpu, oracle, h, bits, "f16", offsets=offsets, ctx="c4 goldens")


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_wide_range_16bit(peat_gpu, oracle, h, dtype):
    """Magnitudes log-uniform over every binade of the format (fp16 30, bf16
    250) with random signs, zeros and subnormals: most elements fall outside
    any window and take the exact path."""
    rng = np.random.default_rng(41)
    n = 1_000_003
    e = rng.integers(0, 31 if dtype == "f16" else 255, n, dtype=np.uint32)
    m = rng.integers(0, 1 << (10 if dtype == "f16" else 7), n, dtype=np.uint32)
    sgn = rng.integers(0, 2, n, dtype=np.uint32)
    bits = ((sgn << 15) | (e << (10 if dtype == "f16" else 7)) | m).astype(np.uint16)
    check(peat_gpu, oracle, h, bits, dtype, ctx="wide")
    offsets = [0, 17, 300_000, 300_000, 999_999, n]
    check(peat_gpu, oracle, h, bits, dtype, offsets=offsets, ctx="wide segmented")


def test_workload_c2_full_against_torch(peat_gpu, h):
    """The [8,2048,4096] bf16 activation: every bf16 value and square is exact in
    binary64, so torch's float64 sums agree to their own rounding."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c2_bf16_rne_vs_rtz(device="cuda")
    r = peat_gpu.peat_tensor_stats(h, w.golden)
    x = w.golden.double().reshape(-1)
    assert r["n"] == r["n_finite"] == x.numel()
    assert math.isclose(r["sum"], float(x.sum()), rel_tol=1e-12, abs_tol=1e-9)
    assert math.isclose(r["sum_sq"], float((x * x).sum()), rel_tol=1e-12)
    assert math.isclose(r["var"], float(x.var(unbiased=False)), rel_tol=1e-10)
    assert r["min"] == float(x.min()) and r["max"] == float(x.max())


def test_one_tensor_bounds_reused_across_calls(peat_gpu, oracle, h):
    """One-tensor calls keep their CTA bounds on the device and rewrite them
    only when the size, alignment, CTA count or stream changes: interleave
    compares and statistics (different CTA counts for the same n), a second
    stream and a misaligned view on one handle."""
    from parity_util import assert_hist_equal, assert_stats_equal
    n = 300_007
    gb, cb = noise_pairs("bf16", n, seed=91)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    ost, ohist = oracle.compare(gb, cb, "bf16", 1e-3, 0.0)
    ots = oracle.tensor_stats(gb, "bf16")
    side = torch.cuda.Stream()
    for rep in range(2):
        st, hist = peat_gpu.peat_compare(h, g, c, 1e-3)
        assert_stats_equal(st, ost, f"compare {rep}")
        assert_hist_equal(hist, ohist, f"compare {rep}")
        check_one(peat_gpu.peat_tensor_stats(h, g), ots, f"stats {rep}")
        st, hist = peat_gpu.peat_compare(h, g, c, 1e-3, stream=side)
        side.synchronize()
        assert_stats_equal(st, ost, f"side stream {rep}")
        st, hist = peat_gpu.peat_compare(h, to_device(gb, "bf16", 3), to_device(cb, "bf16", 3), 1e-3)
        assert_stats_equal(st, ost, f"misaligned {rep}")
        st, hist = peat_gpu.peat_compare(h, g[:n - 5], c[:n - 5], 1e-3)
        o5, _ = oracle.compare(gb[:n - 5], cb[:n - 5], "bf16", 1e-3, 0.0)
        assert_stats_equal(st, o5, f"shorter {rep}")
