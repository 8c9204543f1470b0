"""Fused inject + compare against the two calls it fuses and against the oracle.

peat_inject_compare(golden, models, seed) must give, bit for bit, the
signature of golden against the candidate the injector writes for the same
models and seed; the oracle's compare of golden against the oracle's injected
copy pins both.
"""
import numpy as np
import pytest

from parity_util import assert_hist_equal, assert_stats_equal, noise_pairs, random_pairs, to_device

pytestmark = pytest.mark.gpu

DTYPES = ["f32", "f16", "bf16"]


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0)
    yield handle
    handle.close()


def chains(dtype):
    ms = [
        [dict(kind="rel_gauss", x=1e-3)],
        [dict(kind="add_gauss", x=1e-2)],
        [dict(kind="bias", x=1e-4)],
        [dict(kind="signflip", x=1e-2)],
        [dict(kind="nan_inf", x=1e-3)],
        [dict(kind="rel_gauss", x=1e-3), dict(kind="signflip", x=1e-3), dict(kind="nan_inf", x=1e-4),
         dict(kind="bias", x=-3e-4)],
        [dict(kind="rel_gauss", x=0.5)],                  # large errors: most pairs leave the window
        [dict(kind="signflip", x=1.0)],                   # every element flipped
        [dict(kind="rel_gauss", x=0.0)],                  # candidate == golden
    ]
    if dtype == "f32":
        ms += [[dict(kind=k)] for k in ("cast_f16_rne", "cast_f16_rtz", "cast_bf16_rne", "cast_bf16_rtz")]
        ms += [[dict(kind="rel_gauss", x=1e-4), dict(kind="cast_bf16_rne"), dict(kind="add_gauss", x=1e-6)]]
    return ms


def check(peat, oracle, h, gb, dtype, models, seed, rtol, atol, goff=0, ctx=""):
    g = to_device(gb, dtype, goff)
    fs, fh = peat.peat_inject_compare(h, g, models, seed, rtol, atol)
    # the two calls it fuses, on the GPU
    c, _ = peat.peat_pseudo_error_inject(h, g, models, seed)
    us, uh = peat.peat_compare(h, g, c, rtol, atol)
    assert_stats_equal(fs, us, ctx + " vs unfused")
    assert_hist_equal(fh, uh, ctx + " vs unfused")
    # the oracle's injector and compare
    cb, _ = oracle.inject(gb, dtype, [oracle.model(**m) for m in models], seed)
    os_, oh = oracle.compare(gb, cb, dtype, rtol, atol)
    assert_stats_equal(fs, os_, ctx + " vs oracle")
    assert_hist_equal(fh, oh, ctx + " vs oracle")
    return fs


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("n", [1, 7, 9, 4095, 100003])
def test_fused_matches_inject_then_compare(peat_gpu, oracle, h, dtype, n):
    gb, _ = noise_pairs(dtype, n, seed=300 + n, outliers=min(20, n))
    for models in chains(dtype):
        for seed in (0, 98765432123):
            check(peat_gpu, oracle, h, gb, dtype, models, seed, 1e-3, 0.0, ctx=f"{dtype} n={n} {models} s={seed}")


@pytest.mark.parametrize("dtype", DTYPES)
def test_fused_random_bit_golden(peat_gpu, oracle, h, dtype):
    """Golden of random bit patterns (NaN, Inf, subnormals, every binade):
    the general path with generated candidates, and the rescan beyond the list."""
    n = 300007
    gb, _ = random_pairs(dtype, n, seed=41)
    for models in ([dict(kind="signflip", x=0.3)], [dict(kind="rel_gauss", x=1e-2), dict(kind="nan_inf", x=1e-2)],
                   [dict(kind="add_gauss", x=1.0)]):
        check(peat_gpu, oracle, h, gb, dtype, models, 7, 2.0 ** -7, 1e-6, ctx=f"{dtype} random {models}")


@pytest.mark.parametrize("dtype", DTYPES)
@pytest.mark.parametrize("goff", [1, 3])
def test_fused_misaligned_and_ragged(peat_gpu, oracle, h, dtype, goff):
    n = (1 << 20) + 5
    gb, _ = noise_pairs(dtype, n, seed=77 + goff)
    check(peat_gpu, oracle, h, gb, dtype, [dict(kind="rel_gauss", x=1e-3), dict(kind="nan_inf", x=1e-5)], 11,
          1e-3, 0.0, goff=goff, ctx=f"{dtype} goff={goff}")


def test_fused_playback_snapshot(peat_gpu, oracle, h):
    """A bf16 snapshot of the playback sweep's size class (several tiles per CTA), with the
    sweep's multiplicative noise generated in the kernel."""
    n = (1 << 23) + 129
    gb, _ = noise_pairs("bf16", n, seed=5, rel=0.0, outliers=0)
    check(peat_gpu, oracle, h, gb, "bf16", [dict(kind="rel_gauss", x=1e-4 * 3 ** 0.5)], 5, 2.0 ** -7, 0.0,
          ctx="bf16 playback")


def test_fused_empty_and_rejections(peat_gpu, oracle, h):
    import torch
    g = torch.empty(0, dtype=torch.bfloat16, device="cuda")
    fs, fh = peat_gpu.peat_inject_compare(h, g, [dict(kind="rel_gauss", x=1e-3)], 1, 1e-3)
    os_, oh = oracle.compare(np.zeros(0, np.uint16), np.zeros(0, np.uint16), "bf16", 1e-3, 0.0)
    assert_stats_equal(fs, os_, "empty")
    assert_hist_equal(fh, oh, "empty")
    gb, _ = noise_pairs("bf16", 1000, seed=1)
    g = to_device(gb, "bf16")
    for bad in ([dict(kind="rz", k=3)], [dict(kind="rv", k=3)], [dict(kind="bitflip", k=1, bit_lo=0, bit_hi=3)],
                [], [dict(kind="bias", x=1e-3)] * 9, [dict(kind="cast_f16_rne")], [dict(kind="nan_inf", x=1.5)],
                [dict(kind="add_gauss", x=float("inf"))]):
        with pytest.raises(peat_gpu.PeatError):
            peat_gpu.peat_inject_compare(h, g, bad, 1, 1e-3)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_inject_compare(h, g, [dict(kind="bias", x=1e-3)], 1, -1.0)
    assert "fixed-count" in _err_after(peat_gpu, h, g, [dict(kind="rz", k=3)])
    # the handle still works after the rejections
    check(peat_gpu, oracle, h, gb, "bf16", [dict(kind="bias", x=1e-3)], 2, 1e-3, 0.0, ctx="after rejections")


def _err_after(peat, h, g, models):
    try:
        peat.peat_inject_compare(h, g, models, 1, 1e-3)
    except peat.PeatError as e:
        return str(e)
    return ""
