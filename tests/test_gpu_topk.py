"""GPU parity of the mean of the top errors (Section IV-B-3, "Mean of Top 10%
Errors"): peat_topk_mean through the C ABI against oracle.topk_mean.

Bar: n_finite and k bit-exact; threshold, sum and mean bit-identical (each is
the one binary64 rounding of an exact value on both sides); exact flag set.
"""
import math

import numpy as np
import pytest
import torch

from parity_util import NP_BITS, noise_pairs, random_pairs, to_device

pytestmark = pytest.mark.gpu

DTYPES = ["f32", "f16", "bf16"]
FRACTIONS = [(1, 10), (1, 1), (3, 7), (1, 1000)]
KEYS = ("n_finite", "k", "threshold", "sum", "mean")


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0)
    yield handle
    handle.close()


def check(peat, oracle, h, gb, cb, dtype, num=1, den=10, goff=0, coff=0, ctx=""):
    g, c = to_device(gb, dtype, goff), to_device(cb, dtype, coff)
    gr = peat.peat_topk_mean(h, g, c, num, den)
    orr = oracle.topk_mean(gb, cb, dtype, num, den)
    for k in KEYS:
        assert gr[k] == orr[k], f"{ctx} {dtype} {num}/{den}: {k} gpu={gr[k]!r} oracle={orr[k]!r}"
    assert gr["exact"] == 1, ctx
    return gr


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [0, 1, 7, 4099, 100_003])
def test_random_mixtures(peat_gpu, oracle, h, dtype, n):
    gb, cb = random_pairs(dtype, n, seed=1000 + n)
    for num, den in FRACTIONS:
        check(peat_gpu, oracle, h, gb, cb, dtype, num, den, ctx=f"n={n}")


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("offs", [(1, 1), (1, 0), (3, 5)])
def test_misaligned_bases(peat_gpu, oracle, h, dtype, offs):
    gb, cb = random_pairs(dtype, 50_021, seed=77)
    check(peat_gpu, oracle, h, gb, cb, dtype, goff=offs[0], coff=offs[1], ctx=f"offsets {offs}")


@pytest.mark.parametrize("dtype", DTYPES)
def test_noise_million(peat_gpu, oracle, h, dtype):
    gb, cb = noise_pairs(dtype, (1 << 20) + 3, seed=5)
    for num, den in FRACTIONS:
        check(peat_gpu, oracle, h, gb, cb, dtype, num, den, ctx="noise")


def test_no_finite_pair(peat_gpu, oracle, h):
    n = 10_000
    gb = np.full(n, 0x7FC00000, np.uint32)
    cb = np.arange(n, dtype=np.uint32)
    r = check(peat_gpu, oracle, h, gb, cb, "f32", ctx="all NaN")
    assert r["k"] == 0 and r["mean"] == 0.0
    # a following call on the same handle starts from a clean state
    gb2, cb2 = random_pairs("f32", 9_999, seed=3)
    check(peat_gpu, oracle, h, gb2, cb2, "f32", ctx="after all NaN")


def test_repeated_calls_agree(peat_gpu, oracle, h):
    gb, cb = random_pairs("bf16", 300_001, seed=11)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    a = peat_gpu.peat_topk_mean(h, g, c)
    b = peat_gpu.peat_topk_mean(h, g, c)
    assert a == b


def f32_bits(x):
    return np.asarray(x, np.float32).view(np.uint32)


def test_bucket_ordered_by_the_float32_rounding_error(peat_gpu, oracle, h):
    """Many pairs share RN32(|d|) = 2^24 + 2 with |d| above, on and below it
    (c - g inexact in float32): the k-th largest falls inside that bucket, so
    the exact order of the rounding errors decides which pairs count."""
    rng = np.random.default_rng(8)
    m = 1800  # 3600 listed members: below the 4096 kept for the exact order
    x = rng.random(m).astype(np.float32) * np.float32(0.99)   # in [0, 0.99)
    y = rng.random(m).astype(np.float32) * np.float32(0.99)
    big = np.float32(2 ** 24)
    g = np.concatenate([-x, 2 + y, np.zeros(500, np.float32), np.zeros(10_000, np.float32)])
    c = np.concatenate([np.full(m, big + 2, np.float32), np.full(m, big + 4, np.float32),
                        np.full(500, big + 2, np.float32), rng.random(10_000).astype(np.float32)])
    perm = rng.permutation(g.size)
    gb, cb = f32_bits(g[perm]), f32_bits(c[perm])
    # bucket positions: lo > 0 at 0..1799, lo = 0 at 1800..2299, lo < 0 at 2300..4099
    for num, den in [(1, 10), (1, 7), (1, 4), (3, 10), (1, 1)]:
        check(peat_gpu, oracle, h, gb, cb, "f32", num, den, ctx="bucket")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_overflowing_differences(peat_gpu, oracle, h, dtype):
    """c - g beyond the float32 range (opposite signs near the maximum)."""
    rng = np.random.default_rng(21)
    n = 20_000
    a = (rng.random(n) * 1e38 + 2.3e38).astype(np.float32)
    b = (rng.random(n) * 1e38 + 2.3e38).astype(np.float32)
    sgn = np.where(rng.random(n) < 0.5, 1, -1).astype(np.float32)
    g = a * sgn
    c = np.where(rng.random(n) < 0.3, -b * sgn, g * np.float32(1.0001))
    g[:100], c[:100] = np.float32(3e38), np.float32(-3e38)  # ties in the overflowing range
    if dtype == "f32":
        gb, cb = f32_bits(g), f32_bits(c)
    else:
        gb = (f32_bits(g) >> 16).astype(np.uint16)
        cb = (f32_bits(c) >> 16).astype(np.uint16)
    for num, den in FRACTIONS:
        check(peat_gpu, oracle, h, gb, cb, dtype, num, den, ctx="overflow")


@pytest.mark.parametrize("dtype", DTYPES)
def test_equal_magnitudes(peat_gpu, oracle, h, dtype):
    """All nonzero errors equal: the threshold bucket holds every one of them."""
    n = 65_537
    rng = np.random.default_rng(4)
    gb = np.zeros(n, NP_BITS[dtype])
    one = {"f32": 0x3F800000, "f16": 0x3C00, "bf16": 0x3F80}[dtype]
    cb = np.where(rng.random(n) < 0.5, one, 0).astype(NP_BITS[dtype])
    for num, den in FRACTIONS:
        check(peat_gpu, oracle, h, gb, cb, dtype, num, den, ctx="equal")


def test_workload_c1(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c1_single_fp32(device="cuda")
    gb = w.golden.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)
    cb = w.candidate.cpu().contiguous().view(torch.int32).numpy().view(np.uint32)
    check(peat_gpu, oracle, h, gb, cb, "f32", ctx="c1")


@pytest.mark.parametrize("step", [1, 40])
def test_workload_c5_playback(peat_gpu, oracle, h, step):
    from paper_2609_13544_gb300 import workloads as W
    w = W.PlaybackSweep(n=(1 << 20) + 11, device="cuda").workload(step)
    iv = torch.int32 if w.dtype == "f32" else torch.int16
    gb = w.golden.cpu().contiguous().view(iv).numpy().view(NP_BITS[w.dtype])
    cb = w.candidate.cpu().contiguous().view(iv).numpy().view(NP_BITS[w.dtype])
    check(peat_gpu, oracle, h, gb, cb, w.dtype, ctx=f"c5 step {step}")


def test_c2_full_size_against_torch(peat_gpu, h):
    """[8,2048,4096] bf16 RNE vs RTZ: every |d| is exact in binary64, so torch's
    float64 sort gives the threshold exactly and its float64 sum the total to
    within the accumulation error."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c2_bf16_rne_vs_rtz(device="cuda")
    r = peat_gpu.peat_topk_mean(h, w.golden, w.candidate)
    d = (w.candidate.double() - w.golden.double()).abs().reshape(-1)
    assert r["n_finite"] == d.numel()
    k = math.ceil(d.numel() / 10)
    assert r["k"] == k
    top = torch.topk(d, k, sorted=False).values
    assert r["threshold"] == float(top.min())
    s = float(top.sum())
    assert math.isclose(r["sum"], s, rel_tol=1e-12)
    assert math.isclose(r["mean"], s / k, rel_tol=1e-12)
    assert r["exact"] == 1


def test_inexact_pairs_beyond_the_list(peat_gpu, oracle, h):
    """More than 65536 pairs whose |d| is not a float32 value within 1024
    float32 steps of the k-th largest: the fourth pass sums that range again."""
    rng = np.random.default_rng(31)
    n_near = 100_000
    j = rng.integers(0, 500, n_near)
    c = (np.float32(2 ** 24) + 2 * j).astype(np.float32)           # spacing 2 above 2^24
    g = -(rng.random(n_near).astype(np.float32) * np.float32(0.99) + np.float32(0.005))
    g_rest = np.zeros(400_000, np.float32)
    c_rest = rng.random(400_000).astype(np.float32)
    gb = f32_bits(np.concatenate([g, g_rest]))
    cb = f32_bits(np.concatenate([c, c_rest]))
    perm = rng.permutation(gb.size)
    gb, cb = gb[perm], cb[perm]
    for num, den in [(1, 10), (1, 7), (1, 5), (1, 1)]:
        check(peat_gpu, oracle, h, gb, cb, "f32", num, den, ctx="list overflow")


@pytest.mark.parametrize("num,den", [(1, 20), (1, 10), (3, 40), (1, 7000), (1, 1)])
def test_bucket_beyond_the_list_is_exact(peat_gpu, oracle, h, num, den):
    """More than 65536 inexact pairs tied in float32 with the k-th largest (too
    many to list): the radix passes over their rounding errors resolve the
    m largest exactly, and every field equals the oracle's bit for bit.  The
    rounding errors repeat (g on a coarse grid), so the selected low digit
    holds ties of its own."""
    rng = np.random.default_rng(32)
    m = 70_000
    g = -(rng.integers(1, 3000, m).astype(np.float32) * np.float32(2.0 ** -12))
    c = np.full(m, np.float32(2 ** 24 + 2), np.float32)
    gb = f32_bits(np.concatenate([g, np.zeros(630_000, np.float32)]))
    cb = f32_bits(np.concatenate([c, rng.random(630_000).astype(np.float32)]))
    perm = rng.permutation(gb.size)
    check(peat_gpu, oracle, h, gb[perm], cb[perm], "f32", num, den, ctx="tied bucket")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("pattern", ["every16", "runs"])
def test_sampled_window_misses(peat_gpu, oracle, h, dtype, pattern):
    """Small errors on evenly spaced pairs (every 16th, or the first 256 of
    every 2048) and large ones elsewhere: a sample drawn from such positions
    picks a window that misses the k-th largest, and the exact passes take
    over; either way the result is the oracle's."""
    import torch
    n = 1 << 22
    rng = np.random.default_rng(40)
    g = rng.standard_normal(n).astype(np.float32)
    pos = np.arange(n)
    small = (pos % 16 == 0) if pattern == "every16" else (pos % 2048 < 256)
    rel = np.where(small, 1e-6, 0.3).astype(np.float32)
    c = (g * (1 + rel * rng.standard_normal(n).astype(np.float32))).astype(np.float32)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    iv = torch.int32 if dtype == "f32" else torch.int16
    gb = torch.from_numpy(g).to(tdt).view(iv).numpy().view(NP_BITS[dtype])
    cb = torch.from_numpy(c).to(tdt).view(iv).numpy().view(NP_BITS[dtype])
    for num, den in [(1, 10), (1, 1000)]:
        check(peat_gpu, oracle, h, gb, cb, dtype, num, den, ctx="sample misses")
