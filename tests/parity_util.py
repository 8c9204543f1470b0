"""Helpers shared by the GPU parity tests: input mixtures, oracle fan-out, comparison."""
from __future__ import annotations

import math
import os
from concurrent.futures import ProcessPoolExecutor
import multiprocessing as mp

import numpy as np

NP_BITS = {"f32": np.uint32, "f16": np.uint16, "bf16": np.uint16, "f8e4m3": np.uint8, "f8e5m2": np.uint8}
TORCH_DT = {"f32": "float32", "f16": "float16", "bf16": "bfloat16", "f8e4m3": "float8_e4m3fn",
            "f8e5m2": "float8_e5m2"}
WIDTH = {"f32": 32, "f16": 16, "bf16": 16, "f8e4m3": 8, "f8e5m2": 8}
INT_KEYS = ("n", "count", "n_finite", "argmax_abs", "argmax_rel", "max_ulp", "argmax_ulp")
EXACT_FLOAT_KEYS = ("max_abs", "max_rel", "rtol_eff", "atol_eff", "mean_abs", "var_abs")
SUM_KEYS = ("sum_abs", "sum_sq", "sum_signed")
SUM_RTOL = 1e-10  # the stated bound for the binary64 sums (the design is exact)


def random_pairs(dtype: str, n: int, seed: int):
    """Bit-pattern mixture: close pairs, arbitrary patterns, sign flips, zeros,
    equal values, small values near the subnormal range, and relative noise."""
    rng = np.random.default_rng(seed)
    w = 32 if dtype == "f32" else 16
    top = 2 ** w
    g = rng.integers(0, top, n, dtype=np.uint64)
    # bias towards finite normal numbers of moderate size
    normal = rng.random(n) < 0.6
    if dtype == "f32":
        vals = (rng.standard_normal(n) * np.exp2(rng.integers(-20, 20, n))).astype(np.float32).view(np.uint32)
    elif dtype == "f16":
        vals = (rng.standard_normal(n) * np.exp2(rng.integers(-10, 8, n))).astype(np.float16).view(np.uint16)
    else:
        x = (rng.standard_normal(n) * np.exp2(rng.integers(-30, 30, n))).astype(np.float32)
        vals = (x.view(np.uint32) >> 16).astype(np.uint16)
    g = np.where(normal, vals.astype(np.uint64), g)
    c = g.copy()
    kind = rng.integers(0, 8, n)
    step = rng.integers(-6, 7, n)
    c = np.where(kind <= 2, (g + step.astype(np.uint64)) % top, c)            # close
    c = np.where(kind == 3, rng.integers(0, top, n, dtype=np.uint64), c)      # arbitrary
    sign = np.uint64(1 << (w - 1))
    c = np.where(kind == 4, (g ^ sign), c)                                    # sign flip
    c = np.where(kind == 5, np.uint64(0), c)                                  # zero
    small = rng.integers(0, 2 ** (w // 2), n, dtype=np.uint64)
    g = np.where(kind == 6, small, g)
    c = np.where(kind == 6, small + rng.integers(0, 3, n).astype(np.uint64), c)
    # kind 7: equal
    return g.astype(NP_BITS[dtype]), c.astype(NP_BITS[dtype])


def noise_pairs(dtype: str, n: int, seed: int, rel: float = 1e-3, outliers: int = 20):
    """Realistic recorded-tensor pairs: Gaussian golden, relative noise, a few outliers."""
    import torch
    rng = np.random.default_rng(seed)
    x = rng.standard_normal(n).astype(np.float32)
    y = (x * (1 + rel * rng.standard_normal(n))).astype(np.float32)
    tdt = getattr(torch, TORCH_DT[dtype])
    g = torch.from_numpy(x).to(tdt)
    c = torch.from_numpy(y).to(tdt)
    iv = {"f32": torch.int32}.get(dtype, torch.int16)
    gb = g.view(iv).numpy().view(NP_BITS[dtype]).copy()
    cb = c.view(iv).numpy().view(NP_BITS[dtype]).copy()
    if outliers:
        idx = rng.choice(n, outliers, replace=False)
        cb[idx] = rng.integers(0, 2 ** (8 * cb.itemsize), outliers).astype(cb.dtype)
    return gb, cb


def to_device(bits: np.ndarray, dtype: str, offset: int = 0):
    """Copy bit patterns to a CUDA tensor of the element type, optionally starting
    `offset` elements into a larger allocation (to test misaligned bases)."""
    import torch
    tdt = getattr(torch, TORCH_DT[dtype])
    iv = torch.int32 if dtype == "f32" else torch.int16
    host = torch.from_numpy(bits.view(np.int32 if dtype == "f32" else np.int16).copy())
    buf = torch.empty(bits.size + offset, dtype=iv, device="cuda")
    buf[offset:].copy_(host)
    return buf.view(tdt)[offset:]


def _oracle_chunk(args):
    import oracle
    g, c, off, dtype, rtol, atol = args
    return oracle.compare_segmented(g, c, off, dtype, rtol, atol)


def oracle_segmented(g, c, offsets, dtype, rtol, atol, workers: int | None = None):
    """The oracle over many segments, fanned out to spawned processes."""
    import oracle
    offsets = np.asarray(offsets, np.int64)
    nseg = offsets.size - 1
    total = int(offsets[-1])
    if workers is None:
        workers = min(16, os.cpu_count() or 1)
    if total < 2_000_000 or workers <= 1 or nseg < 2:
        return oracle.compare_segmented(g, c, offsets, dtype, rtol, atol)
    # contiguous chunks of segments with about equal element counts
    target = total / (workers * 2)
    cuts = [0]
    acc = 0
    for s in range(nseg):
        acc += int(offsets[s + 1] - offsets[s])
        if acc >= target and s + 1 < nseg:
            cuts.append(s + 1)
            acc = 0
    cuts.append(nseg)
    jobs = []
    for a, b in zip(cuts[:-1], cuts[1:]):
        lo, hi = int(offsets[a]), int(offsets[b])
        jobs.append((g[lo:hi], c[lo:hi], offsets[a:b + 1] - lo, dtype, rtol, atol))
    ctx = mp.get_context("spawn")
    with ProcessPoolExecutor(max_workers=workers, mp_context=ctx) as ex:
        parts = list(ex.map(_oracle_chunk, jobs))
    stats = [s for p in parts for s in p[0]]
    hist = np.concatenate([p[1] for p in parts]) if parts else np.zeros((0, 2, 64), np.uint64)
    return stats, hist


def close_sum(a: float, b: float) -> bool:
    if a == b:
        return True
    return abs(a - b) <= SUM_RTOL * abs(b)


def assert_stats_equal(gs: dict, os_: dict, ctx=""):
    for k in INT_KEYS:
        assert gs[k] == os_[k], f"{ctx}: {k} gpu={gs[k]} oracle={os_[k]}"
    for k in EXACT_FLOAT_KEYS:
        assert gs[k] == os_[k], f"{ctx}: {k} gpu={gs[k]!r} oracle={os_[k]!r}"
    for k in SUM_KEYS:
        assert close_sum(gs[k], os_[k]), f"{ctx}: {k} gpu={gs[k]!r} oracle={os_[k]!r}"


def assert_hist_equal(gh, oh, ctx=""):
    gh = np.asarray(gh)
    oh = np.asarray(oh)
    if not np.array_equal(gh, oh):
        bad = np.argwhere(gh != oh)
        raise AssertionError(f"{ctx}: histogram differs at {bad[:10].tolist()} gpu={gh[tuple(bad[0])]} "
                             f"oracle={oh[tuple(bad[0])]}")


def f64_pairs(n: int, seed: int):
    """binary64 mixture: relative noise, one-ULP neighbours, arbitrary patterns,
    sign flips, zeros, subnormals, operands near the largest double (their
    difference overflows) and equal pairs."""
    rng = np.random.default_rng(seed)
    g = (rng.standard_normal(n) * np.exp2(rng.integers(-60, 60, n))).astype(np.float64)
    c = g * (1 + 1e-12 * rng.standard_normal(n))
    kind = rng.integers(0, 9, n)
    gb, cb = g.view(np.uint64).copy(), c.view(np.uint64).copy()
    cb = np.where(kind == 0, gb + rng.integers(-3, 4, n).astype(np.int64).astype(np.uint64), cb)
    cb = np.where(kind == 1, rng.integers(0, 2 ** 63, n, dtype=np.uint64) * np.uint64(2)
                  + rng.integers(0, 2, n, dtype=np.uint64), cb)
    cb = np.where(kind == 2, gb ^ np.uint64(1 << 63), cb)
    cb = np.where(kind == 3, np.uint64(0), cb)
    sub = rng.integers(0, 1 << 52, n, dtype=np.uint64)
    gb = np.where(kind == 4, sub, gb)
    cb = np.where(kind == 4, sub + rng.integers(0, 5, n, dtype=np.uint64), cb)
    big = np.float64(1.7e308)
    gb = np.where(kind == 5, np.array([-big]).view(np.uint64)[0], gb)
    cb = np.where(kind == 5, (big * (1 - 1e-3 * rng.random(n))).view(np.uint64), cb)
    cb = np.where(kind == 6, gb, cb)
    return gb.astype(np.uint64), cb.astype(np.uint64)
