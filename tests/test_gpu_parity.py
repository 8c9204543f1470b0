"""GPU parity: the CUDA path through the C ABI against the oracle, element by element.

Bar: every integer output bit-exact (counts, histograms, argmax indices, ULP
maxima), max_abs/max_rel and the effective tolerances bit-identical, the
three binary64 sums within 1e-10 relative (the design is exact, so they are
expected bit-identical as well).
"""
import math

import numpy as np
import pytest

from parity_util import (assert_hist_equal, assert_stats_equal, noise_pairs, oracle_segmented, random_pairs,
                         to_device)

pytestmark = pytest.mark.gpu

DTYPES = ["f32", "f16", "bf16"]


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0, max_segments=70000)
    yield handle
    handle.close()


def run_pair(peat, h, gb, cb, dtype, rtol, atol, goff=0, coff=0):
    g = to_device(gb, dtype, goff)
    c = to_device(cb, dtype, coff)
    return peat.peat_compare(h, g, c, rtol, atol)


def check_pair(peat, oracle, h, gb, cb, dtype, rtol, atol, goff=0, coff=0, ctx=""):
    gs, gh = run_pair(peat, h, gb, cb, dtype, rtol, atol, goff, coff)
    os_, oh = oracle.compare(gb, cb, dtype, rtol, atol)
    assert_stats_equal(gs, os_, ctx)
    assert_hist_equal(gh, oh, ctx)
    return gs


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [0, 1, 7, 8, 9, 4095, 100003])
def test_random_pairs(peat_gpu, oracle, h, dtype, n):
    gb, cb = random_pairs(dtype, n, seed=1000 + n)
    check_pair(peat_gpu, oracle, h, gb, cb, dtype, 1e-3, 0.0, ctx=f"{dtype} n={n}")
    check_pair(peat_gpu, oracle, h, gb, cb, dtype, 2.0 ** -7, 1e-6, ctx=f"{dtype} n={n} atol")


@pytest.mark.parametrize("dtype", DTYPES)
def test_noise_ragged_large(peat_gpu, oracle, h, dtype):
    n = (1 << 20) + 3
    gb, cb = noise_pairs(dtype, n, seed=7, rel=1e-3)
    check_pair(peat_gpu, oracle, h, gb, cb, dtype, 1e-3, 0.0, ctx=f"{dtype} noise")


@pytest.mark.parametrize("dtype", DTYPES)
def test_general_pairs_beyond_the_list(peat_gpu, oracle, h, dtype):
    """Random bit patterns: most pairs leave the window, so every CTA piece
    holds more general pairs than its list (16384) and is rescanned."""
    n = 12_000_017
    gb, cb = random_pairs(dtype, n, seed=4242)
    check_pair(peat_gpu, oracle, h, gb, cb, dtype, 1e-3, 0.0, ctx=f"{dtype} rescan")


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("offs", [(1, 1), (3, 3), (1, 2), (0, 5)])
def test_misaligned_bases(peat_gpu, oracle, h, dtype, offs):
    gb, cb = noise_pairs(dtype, 50021, seed=11, rel=1e-2)
    check_pair(peat_gpu, oracle, h, gb, cb, dtype, 1e-2, 0.0, goff=offs[0], coff=offs[1], ctx=f"{dtype} {offs}")


@pytest.mark.parametrize("dtype", DTYPES)
def test_segmented_random_layout(peat_gpu, oracle, h, dtype):
    rng = np.random.default_rng(5)
    sizes = rng.choice([0, 1, 2, 7, 64, 1000, 4097, 30000], size=400)
    off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)
    n = int(off[-1])
    gb, cb = random_pairs(dtype, n, seed=77)
    g, c = to_device(gb, dtype), to_device(cb, dtype)
    gs, gh = peat_gpu.peat_compare_segmented(h, g, c, off, 1e-3, 0.0)
    os_, oh = oracle_segmented(gb, cb, off, dtype, 1e-3, 0.0)
    assert len(gs) == len(os_) == 400
    for s in range(400):
        assert_stats_equal(gs[s], os_[s], f"{dtype} seg {s}")
    assert_hist_equal(gh, oh, dtype)


@pytest.mark.parametrize("dtype", DTYPES)
def test_edge_tensors(peat_gpu, oracle, h, dtype):
    n = 4099
    nan = {"f32": 0x7FC00000, "f16": 0x7E00, "bf16": 0x7FC0}[dtype]
    inf = {"f32": 0x7F800000, "f16": 0x7C00, "bf16": 0x7F80}[dtype]
    one = {"f32": 0x3F800000, "f16": 0x3C00, "bf16": 0x3F80}[dtype]
    neg0 = {"f32": 0x80000000, "f16": 0x8000, "bf16": 0x8000}[dtype]
    T = np.uint32 if dtype == "f32" else np.uint16
    cases = {
        "all_nan": (np.full(n, nan, T), np.full(n, nan, T)),
        "nan_vs_one": (np.full(n, nan, T), np.full(n, one, T)),
        "all_equal": (np.full(n, one, T), np.full(n, one, T)),
        "all_inf": (np.full(n, inf, T), np.full(n, inf, T)),
        "zero_vs_negzero": (np.zeros(n, T), np.full(n, neg0, T)),
        "inf_vs_neg": (np.full(n, inf, T), np.full(n, inf | neg0, T)),
    }
    for name, (gb, cb) in cases.items():
        check_pair(peat_gpu, oracle, h, gb, cb, dtype, 1e-3, 0.0, ctx=f"{dtype} {name}")


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_sweep_every_candidate_pattern(peat_gpu, oracle, h, dtype):
    """For 96 golden values spread over all exponents and both signs, every one of
    the 65,536 candidate bit patterns (6.3M pairs)."""
    rng = np.random.default_rng(9)
    mb = 10 if dtype == "f16" else 7
    nexp = 32 if dtype == "f16" else 256
    exps = np.linspace(0, nexp - 1, 48).astype(np.uint32)
    gl = []
    for s in (0, 1):
        for e in exps:
            gl.append((s << 15) | (int(e) << mb) | int(rng.integers(0, 1 << mb)))
    goldens = np.array(gl, np.uint16)
    cand = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    gb = np.repeat(goldens, 65536)
    cb = np.tile(cand, goldens.size)
    off = np.arange(goldens.size + 1, dtype=np.int64) * 65536
    g, c = to_device(gb, dtype), to_device(cb, dtype)
    gs, gh = peat_gpu.peat_compare_segmented(h, g, c, off, 2.0 ** -7, 0.0)
    os_, oh = oracle_segmented(gb, cb, off, dtype, 2.0 ** -7, 0.0)
    for s in range(goldens.size):
        assert_stats_equal(gs[s], os_[s], f"{dtype} golden {hex(goldens[s])}")
    assert_hist_equal(gh, oh, dtype)


def test_determinism(peat_gpu, h):
    import torch
    gb, cb = noise_pairs("bf16", 3_000_001, seed=3)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    stats = [torch.empty(160, dtype=torch.uint8, device="cuda") for _ in range(3)]
    hists = [torch.empty(128, dtype=torch.int64, device="cuda") for _ in range(3)]
    for s, hh in zip(stats, hists):
        peat_gpu.peat_compare_raw(h, g, c, 1e-3, 0.0, s, hh)
    torch.cuda.synchronize()
    for s, hh in zip(stats[1:], hists[1:]):
        assert torch.equal(s, stats[0]) and torch.equal(hh, hists[0])


def test_invalid_arguments(peat_gpu, h):
    import torch
    g = torch.zeros(10, device="cuda")
    s = torch.empty(160, dtype=torch.uint8, device="cuda")
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_compare_raw(h, g, g, -1.0, 0.0, s)
    assert e.value.status == 1
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_compare_segmented_raw(h, g, g, [0, 5, 3, 10], 0.0, 0.0, s)
    assert e.value.status == 1
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_compare_segmented_raw(h, g, g, [1, 10], 0.0, 0.0, s)
    assert e.value.status == 1
    small = peat_gpu.Handle(0, max_segments=2)
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_compare_segmented_raw(small, g, g, [0, 1, 2, 10], 0.0, 0.0, s)
    assert e.value.status == 2
    small.close()


def test_forced_wait_expiry_reports_timeout_and_context_survives(peat_gpu, oracle, h):
    """The pipeline's bounded waits: with the test flag every wait gives up at
    once; the kernel drains its copies, returns, and the next call on that
    handle reports PEAT_ERR_TIMEOUT.  The GPU context stays usable."""
    import torch
    gb, cb = noise_pairs("bf16", 1_000_003, seed=17)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    s = torch.empty(160, dtype=torch.uint8, device="cuda")
    bad = peat_gpu.Handle(0, flags=peat_gpu.PEAT_FLAG_TEST_EXPIRE_WAITS)
    peat_gpu.peat_compare_raw(bad, g, c, 1e-3, 0.0, s)
    torch.cuda.synchronize()
    with pytest.raises(peat_gpu.PeatError) as e:
        peat_gpu.peat_compare_raw(bad, g, c, 1e-3, 0.0, s)
    assert e.value.status == 5
    torch.cuda.synchronize()
    bad.close()
    check_pair(peat_gpu, oracle, h, gb, cb, "bf16", 1e-3, 0.0, ctx="after forced expiry")


@pytest.mark.parametrize("rtol", [2.0 ** -7, 2.0 ** -3, 1e-3])
@pytest.mark.parametrize("atol", [0.0, 1e-7])
def test_tolerance_ties_float32(peat_gpu, oracle, h, rtol, atol):
    """Pairs whose |c - g| is the float32 rounding of rtol |g| exactly, and their
    one-step neighbours: the tolerance decided at and around the tie (with
    atol = 0 by the sign of rtol |g| - |d| in the window path)."""
    rng = np.random.default_rng(61)
    n = 200_000
    mag = (rng.standard_normal(n) * np.exp2(rng.integers(-30, 30, n))).astype(np.float32)
    g = (mag.view(np.uint32) & np.uint32(0xFFFFF000)).view(np.float32)  # low mantissa bits clear
    r32 = np.float32(rtol)
    a = (np.abs(g).astype(np.float64) * np.float64(r32)).astype(np.float32)  # RN32(rtol |g|)
    c0 = (g + np.where(rng.random(n) < 0.5, a, -a)).astype(np.float32)
    up = np.nextafter(c0, np.float32(np.inf))
    dn = np.nextafter(c0, np.float32(-np.inf))
    gb = np.concatenate([g, g, g]).view(np.uint32)
    cb = np.concatenate([c0, up, dn]).view(np.uint32)
    perm = rng.permutation(gb.size)
    gs = check_pair(peat_gpu, oracle, h, gb[perm], cb[perm], "f32", rtol, atol, ctx=f"ties rtol={rtol} atol={atol}")
    assert gs["within_tol"] > 0 and gs["mismatch"] > 0


@pytest.mark.parametrize("case", ["cancel_f32", "overflow_f64", "mixed_f64", "subnormal_var_f64", "bf16_many"])
def test_mean_var_edges_match_the_oracle(peat_gpu, oracle, h, case):
    """The Mean and Variance of Errors scores at their edges, bit for bit: a
    variance far below mean^2, |d| past the largest double (mean +inf), a
    variance past it, a variance on the subnormal grid, and a long bf16 run
    (many digits of the exact sums in use)."""
    import torch
    big = np.finfo(np.float64).max
    if case == "cancel_f32":
        g, c, dt = np.zeros(3, np.float32), (1 + np.arange(3) * 2.0 ** -23).astype(np.float32), "f32"
    elif case == "overflow_f64":
        g, c, dt = np.array([-big, -big]), np.array([big, big]), "f64"
    elif case == "mixed_f64":
        g, c, dt = np.array([-big, 0.0, 1.0]), np.array([big, 0.0, 1.0 + 2.0 ** -52]), "f64"
    elif case == "subnormal_var_f64":
        g, c, dt = np.zeros(3), np.array([3 * 2.0 ** -520, 0.0, 2.0 ** -520]), "f64"
    else:
        gb, cb = noise_pairs("bf16", 3_000_017, seed=91)
        g, c, dt = gb, cb, "bf16"
    if dt == "bf16":
        gt, ct = to_device(g, "bf16"), to_device(c, "bf16")
        gbits, cbits = g, c
    else:
        gt, ct = torch.from_numpy(g).cuda(), torch.from_numpy(c).cuda()
        gbits, cbits = g.view(np.uint32 if dt == "f32" else np.uint64), c.view(np.uint32 if dt == "f32" else np.uint64)
    st, hist = peat_gpu.peat_compare(h, gt, ct, 1e-3, 0.0)
    ost, oh = oracle.compare(gbits, cbits, dt, 1e-3, 0.0)
    assert_stats_equal(st, ost, case)
    assert (st["mean_abs"], st["var_abs"]) == (ost["mean_abs"], ost["var_abs"])
