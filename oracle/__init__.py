"""The oracle: a plain, slow, exact CPU statement of the PEAT error signature.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s ``cpu_baseline`` leg may import this package.  It shares no
code with the CUDA library in ``paper_2609_13544_gb300`` and imports nothing
from it.

Everything is computed by ``peat_oracle.c`` (see its header comment for the
definitions, which follow Section IV-B-3 "FI Assessment Scores" and the Err
step of Alg. 1 / Alg. 2).  This module marshals numpy arrays, and forms the
last exact step of a few scores with Python integers and ``Fraction``: the
mean and variance of |d| from the C code's exact sums, and the context
statistics' mean and variance.
"""
from __future__ import annotations

import ctypes
from typing import Sequence

import numpy as np

from .build import LIB, build

DTYPES = {"f32": 0, "f16": 1, "bf16": 2, "f8e4m3": 3, "f8e5m2": 4, "f64": 5}
ITEMSIZE = {"f32": 4, "f16": 2, "bf16": 2, "f8e4m3": 1, "f8e5m2": 1, "f64": 8}
CLASSES = ("exact", "within_tol", "mismatch", "nan_inf_asym", "sign_flip")
INJECT_KINDS = {
    "rz": 0, "rv": 1, "bitflip": 2, "nan_inf": 3, "signflip": 4, "rel_gauss": 5,
    "add_gauss": 6, "bias": 7, "cast_f16_rne": 8, "cast_f16_rtz": 9, "cast_bf16_rne": 10,
    "cast_bf16_rtz": 11,
}


class Stats(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_uint64),
        ("count", ctypes.c_uint64 * 5),
        ("n_finite", ctypes.c_uint64),
        ("max_abs", ctypes.c_double),
        ("argmax_abs", ctypes.c_int64),
        ("max_rel", ctypes.c_double),
        ("argmax_rel", ctypes.c_int64),
        ("max_ulp", ctypes.c_uint64),
        ("argmax_ulp", ctypes.c_int64),
        ("sum_abs", ctypes.c_double),
        ("sum_sq", ctypes.c_double),
        ("sum_signed", ctypes.c_double),
        ("rtol_eff", ctypes.c_double),
        ("atol_eff", ctypes.c_double),
    ]


class TopK(ctypes.Structure):
    _fields_ = [
        ("n_finite", ctypes.c_uint64),
        ("k", ctypes.c_uint64),
        ("threshold", ctypes.c_double),
        ("sum", ctypes.c_double),
        ("mean", ctypes.c_double),
    ]


ACC_WORDS, ACC_LSB = 72, -2304


class TStats(ctypes.Structure):
    _fields_ = [
        ("n", ctypes.c_uint64),
        ("n_finite", ctypes.c_uint64),
        ("n_nan", ctypes.c_uint64),
        ("n_inf", ctypes.c_uint64),
        ("min", ctypes.c_double),
        ("max", ctypes.c_double),
        ("sum_words", ctypes.c_uint64 * ACC_WORDS),
        ("sum_sq_words", ctypes.c_uint64 * ACC_WORDS),
    ]


class InjectModel(ctypes.Structure):
    _fields_ = [
        ("kind", ctypes.c_int32),
        ("k", ctypes.c_int32),
        ("bit_lo", ctypes.c_int32),
        ("bit_hi", ctypes.c_int32),
        ("x", ctypes.c_double),
    ]


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        path = build()
        L = ctypes.CDLL(str(path))
        vp, i64, i32, dbl = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
        L.orc_compare.argtypes = [vp, vp, i64, i32, dbl, dbl, ctypes.POINTER(Stats), vp]
        L.orc_compare.restype = i32
        L.orc_compare_segmented.argtypes = [vp, vp, vp, i64, i32, dbl, dbl, ctypes.POINTER(Stats), vp]
        L.orc_compare_segmented.restype = i32
        L.orc_compare_segmented_sums.argtypes = [vp, vp, vp, i64, i32, dbl, dbl, ctypes.POINTER(Stats), vp, vp]
        L.orc_compare_segmented_sums.restype = i32
        L.orc_topk_mean.argtypes = [vp, vp, i64, i32, ctypes.c_uint64, ctypes.c_uint64, ctypes.POINTER(TopK)]
        L.orc_topk_mean.restype = i32
        L.orc_tensor_stats.argtypes = [vp, i64, i32, ctypes.POINTER(TStats)]
        L.orc_tensor_stats.restype = i32
        L.orc_ulp_key.argtypes = [ctypes.c_uint64, i32]
        L.orc_ulp_key.restype = i64
        L.orc_exact_sum.argtypes = [vp, i64]
        L.orc_exact_sum.restype = dbl
        L.orc_exact_dot.argtypes = [vp, vp, i64]
        L.orc_exact_dot.restype = dbl
        L.orc_inject.argtypes = [vp, vp, i64, i32, ctypes.POINTER(InjectModel), i32, ctypes.c_uint64, vp]
        L.orc_inject.restype = i32
        L.orc_philox4x32_10.argtypes = [vp, vp, vp]
        L.orc_philox4x32_10.restype = None
        L.orc_normal_pair_from_words.argtypes = [ctypes.c_uint32, ctypes.c_uint32, vp]
        L.orc_normal_pair_from_words.restype = None
        L.orc_sin2pi.argtypes = [ctypes.c_float]
        L.orc_sin2pi.restype = ctypes.c_float
        L.orc_logf.argtypes = [ctypes.c_float]
        L.orc_logf.restype = ctypes.c_float
        L.orc_cos2pi.argtypes = [ctypes.c_float]
        L.orc_cos2pi.restype = ctypes.c_float
        _lib = L
    return _lib


def _bits(x, dtype: str) -> np.ndarray:
    """Raw bit patterns of x as a contiguous uint8/uint16/uint32 array."""
    size = ITEMSIZE[dtype]
    if hasattr(x, "detach"):  # a CPU torch tensor (bf16 and fp8 have no numpy dtype)
        import torch
        x = x.detach().cpu().contiguous()
        x = x.view({8: torch.int64, 4: torch.int32, 2: torch.int16, 1: torch.uint8}[size]).numpy()
    x = np.ascontiguousarray(x)
    if x.dtype.itemsize != size:
        raise ValueError(f"{dtype} needs {size}-byte elements, got {x.dtype}")
    return x.reshape(-1).view({8: np.uint64, 4: np.uint32, 2: np.uint16, 1: np.uint8}[size])


def _stats_dict(s: Stats) -> dict:
    d = {f: getattr(s, f) for f, _ in Stats._fields_ if f != "count"}
    d["count"] = [int(v) for v in s.count]
    for name, v in zip(CLASSES, s.count):
        d[name] = int(v)
    return d


def compare(g, c, dtype: str, rtol: float, atol: float = 0.0):
    """Signature of one tensor pair: (stats dict, hist uint64[2, 64])."""
    gb, cb = _bits(g, dtype), _bits(c, dtype)
    if gb.size != cb.size:
        raise ValueError("golden and candidate differ in length")
    stats, hist = compare_segmented(gb, cb, [0, gb.size], dtype, rtol, atol)
    return stats[0], hist[0]


def mean_var(S1, S2, n_finite: int) -> tuple:
    """The Mean and Variance of Errors scores (Section IV-B-3) over the n_f
    finite pairs, from the exact sums S1 = sum |d| and S2 = sum d^2
    (Fractions): mean = S1 / n_f and var = (n_f S2 - S1^2) / n_f^2
    (population variance), each the exact rational rounded once
    (float(Fraction) rounds to nearest even; past the largest double: inf)."""
    if n_finite == 0:
        return 0.0, 0.0
    nf = int(n_finite)
    return _rn(S1 / nf), _rn((nf * S2 - S1 * S1) / (nf * nf))


def _rn(q) -> float:
    """RN-even binary64 of a non-negative rational, +inf past the largest double."""
    try:
        return float(q)
    except OverflowError:
        return float("inf")


def topk_mean(g, c, dtype: str, num: int = 1, den: int = 10) -> dict:
    """Mean of the ceil(n_finite * num / den) largest |c - g| (Section IV-B-3,
    "Mean of Top 10% Errors"): dict of n_finite, k, threshold, sum, mean."""
    gb, cb = _bits(g, dtype), _bits(c, dtype)
    if gb.size != cb.size:
        raise ValueError("golden and candidate differ in length")
    out = TopK()
    rc = lib().orc_topk_mean(gb.ctypes.data, cb.ctypes.data, gb.size, DTYPES[dtype], num, den, ctypes.byref(out))
    if rc:
        raise ValueError(f"oracle rejected the arguments (code {rc})")
    return {f: getattr(out, f) for f, _ in TopK._fields_}


def isclose_grid(g, c, dtype: str, rtols, atols) -> np.ndarray:
    """torch.isclose pass counts over a tolerance grid (Section III-A, Fig. 5):
    cell (i, j) = EXACT + WITHIN_TOL of the compare with (rtols[i], atols[j])."""
    out = np.zeros((len(rtols), len(atols)), np.uint64)
    for i, r in enumerate(rtols):
        for j, a in enumerate(atols):
            st, _ = compare(g, c, dtype, float(r), float(a))
            out[i, j] = st["exact"] + st["within_tol"]
    return out


def _acc_int(words) -> int:
    """The fixed-point words as a Python integer (value = integer * 2^ACC_LSB)."""
    v = 0
    for j, w in enumerate(words):
        v |= int(w) << (64 * j)
    if v >> (64 * ACC_WORDS - 1):
        v -= 1 << (64 * ACC_WORDS)
    return v


def tensor_stats(x, dtype: str) -> dict:
    """Context statistics of one tensor (Section IV-C-2): counts, finite min and
    max, and sum, sum of squares, mean and population variance of the finite
    elements, each the exact value rounded once (Python integers and
    correctly rounded integer division carry the last steps)."""
    from fractions import Fraction
    xb = _bits(x, dtype)
    out = TStats()
    rc = lib().orc_tensor_stats(xb.ctypes.data, xb.size, DTYPES[dtype], ctypes.byref(out))
    if rc:
        raise ValueError(f"oracle rejected the arguments (code {rc})")
    s1, s2, nf = _acc_int(out.sum_words), _acc_int(out.sum_sq_words), out.n_finite
    unit = 1 << (-ACC_LSB)
    d = {"n": out.n, "n_finite": nf, "n_nan": out.n_nan, "n_inf": out.n_inf,
         "sum": float(Fraction(s1, unit)), "sum_sq": float(Fraction(s2, unit)),
         "mean": float(Fraction(s1, nf * unit)) if nf else 0.0,
         "var": float(Fraction(nf * s2 * unit - s1 * s1, nf * nf * unit * unit)) if nf else 0.0,
         "min": out.min, "max": out.max}
    return d


def tensor_stats_segmented(x, offsets: Sequence[int], dtype: str) -> list:
    xb = _bits(x, dtype)
    return [tensor_stats(xb[int(offsets[s]):int(offsets[s + 1])], dtype) for s in range(len(offsets) - 1)]


def _exact_ranks(v):
    """Ranks 1..n of the values, ties taking the mean of the ranks they span."""
    from fractions import Fraction
    n = len(v)
    order = sorted(range(n), key=lambda i: v[i])
    r = [Fraction(0)] * n
    i = 0
    while i < n:
        j = i
        while j + 1 < n and v[order[j + 1]] == v[order[i]]:
            j += 1
        for k in range(i, j + 1):
            r[order[k]] = Fraction(i + j + 2, 2)
        i = j + 1
    return r


def spearman(x, y) -> float:
    """Spearman rank correlation (Section IV-C-2): Pearson correlation of the
    ranks (mean ranks for ties), exact up to one square root taken at 60
    significant digits; NaN when n < 2 or a ranking is constant."""
    from decimal import Decimal, localcontext
    x, y = [float(a) for a in x], [float(b) for b in y]
    n = len(x)
    if n != len(y):
        raise ValueError("x and y differ in length")
    if n < 2:
        return float("nan")
    rx, ry = _exact_ranks(x), _exact_ranks(y)
    mx, my = sum(rx) / n, sum(ry) / n
    cxy = sum((a - mx) * (b - my) for a, b in zip(rx, ry))
    cxx = sum((a - mx) ** 2 for a in rx)
    cyy = sum((b - my) ** 2 for b in ry)
    if cxx == 0 or cyy == 0:
        return float("nan")
    with localcontext() as ctx:
        ctx.prec = 60
        q = (Decimal(cxy.numerator) / Decimal(cxy.denominator)) / (
            (Decimal(cxx.numerator) / Decimal(cxx.denominator)) * (Decimal(cyy.numerator) / Decimal(cyy.denominator))).sqrt()
        return float(q)


def mean_std(x, ddof: int = 0):
    """Model-wise error range of one layer (Section IV-C-1): mean and standard
    deviation of its scores across epochs (ddof 0: population, 1: sample),
    exact up to one square root at 60 significant digits."""
    from decimal import Decimal, localcontext
    from fractions import Fraction
    v = [Fraction(float(a)) for a in x]
    n = len(v)
    if n == 0:
        return float("nan"), float("nan")
    m = sum(v) / n
    if n <= ddof:
        return float(m), float("nan")
    var = sum((a - m) ** 2 for a in v) / (n - ddof)
    with localcontext() as ctx:
        ctx.prec = 60
        sd = (Decimal(var.numerator) / Decimal(var.denominator)).sqrt()
    return float(m), float(sd)


def trend(x, y) -> dict:
    """The cross-step trend of a score over replayed epochs (Alg. 1's Err step
    per recorded epoch, read across epochs as in Section IV-C-1): the
    least-squares line log y = intercept + slope log x through the points with
    x, y finite and positive.  math.log per point, then the normal equations
    in exact rationals on those logs, each result rounded once."""
    import math
    from fractions import Fraction
    pts = [(math.log(float(a)), math.log(float(b))) for a, b in zip(x, y)
           if math.isfinite(a) and math.isfinite(b) and a > 0 and b > 0]
    out = {"slope": float("nan"), "intercept": float("nan"), "r2": float("nan"), "used": len(pts)}
    m = len(pts)
    if m < 2:
        return out
    lx = [Fraction(a) for a, _ in pts]
    ly = [Fraction(b) for _, b in pts]
    mx, my = sum(lx) / m, sum(ly) / m
    sxx = sum((a - mx) ** 2 for a in lx)
    if sxx == 0:
        return out
    sxy = sum((a - mx) * (b - my) for a, b in zip(lx, ly))
    syy = sum((b - my) ** 2 for b in ly)
    slope = sxy / sxx
    out["slope"], out["intercept"] = float(slope), float(my - slope * mx)
    if syy != 0:
        out["r2"] = float(1 - (syy - slope * sxy) / syy)  # the residual sum of squares is syy - slope sxy
    return out


def compare_segmented(g, c, offsets: Sequence[int], dtype: str, rtol: float, atol: float = 0.0):
    """Per-segment signatures: (list of stats dicts, hist uint64[nseg, 2, 64])."""
    gb, cb = _bits(g, dtype), _bits(c, dtype)
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    nseg = off.size - 1
    if gb.size != cb.size or nseg < 0 or (nseg >= 0 and off[-1] > gb.size):
        raise ValueError("bad offsets or lengths")
    st = (Stats * max(nseg, 1))()
    hist = np.zeros((max(nseg, 1), 2, 64), np.uint64)
    words = np.zeros((max(nseg, 1), 2, ACC_WORDS), np.uint64)
    rc = lib().orc_compare_segmented_sums(gb.ctypes.data, cb.ctypes.data, off.ctypes.data, nseg,
                                          DTYPES[dtype], rtol, atol, st, hist.ctypes.data, words.ctypes.data)
    if rc:
        raise ValueError(f"oracle rejected the arguments (code {rc})")
    from fractions import Fraction
    unit = 1 << (-ACC_LSB)
    out = []
    for s in range(nseg):
        d = _stats_dict(st[s])
        # the exact sums themselves (they let a caller combine segments exactly)
        d["S1_exact"] = Fraction(_acc_int(words[s, 0]), unit)
        d["S2_exact"] = Fraction(_acc_int(words[s, 1]), unit)
        d["mean_abs"], d["var_abs"] = mean_var(d["S1_exact"], d["S2_exact"], d["n_finite"])
        out.append(d)
    return out, hist[:nseg]


def ulp_key(bits: int, dtype: str) -> int:
    return int(lib().orc_ulp_key(int(bits), DTYPES[dtype]))


def exact_sum(x) -> float:
    x = np.ascontiguousarray(x, np.float64)
    return float(lib().orc_exact_sum(x.ctypes.data, x.size))


def exact_dot(x, y) -> float:
    x = np.ascontiguousarray(x, np.float64)
    y = np.ascontiguousarray(y, np.float64)
    return float(lib().orc_exact_dot(x.ctypes.data, y.ctypes.data, x.size))


def model(kind: str, k: int = 0, bit_lo: int = 0, bit_hi: int = 0, x: float = 0.0) -> dict:
    return {"kind": kind, "k": k, "bit_lo": bit_lo, "bit_hi": bit_hi, "x": x}


def inject(src, dtype: str, models: Sequence[dict], seed: int):
    """Apply the error models in order; returns (dst bits array, counts uint64[nmodels])."""
    sb = _bits(src, dtype)
    dst = np.empty_like(sb)
    arr = (InjectModel * max(len(models), 1))()
    for i, m in enumerate(models):
        arr[i] = InjectModel(INJECT_KINDS[m["kind"]], m.get("k", 0), m.get("bit_lo", 0),
                             m.get("bit_hi", 0), m.get("x", 0.0))
    counts = np.zeros(max(len(models), 1), np.uint64)
    rc = lib().orc_inject(dst.ctypes.data, sb.ctypes.data, sb.size, DTYPES[dtype], arr, len(models),
                          ctypes.c_uint64(seed), counts.ctypes.data)
    if rc:
        raise ValueError(f"oracle rejected the arguments (code {rc})")
    return dst, counts[: len(models)]


def philox(ctr: Sequence[int], key: Sequence[int]) -> list:
    c = np.array(ctr, np.uint32)
    k = np.array(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(c.ctypes.data, k.ctypes.data, out.ctypes.data)
    return [int(v) for v in out]


def normal_pair_from_words(w0: int, w1: int) -> tuple:
    """The Box-Muller pair (r cos 2 pi u2, r sin 2 pi u2) of two Philox words."""
    z = np.zeros(2, np.float32)
    lib().orc_normal_pair_from_words(w0, w1, z.ctypes.data)
    return float(z[0]), float(z[1])


def logf(x: float) -> float:
    return float(lib().orc_logf(x))


def cos2pi(u: float) -> float:
    return float(lib().orc_cos2pi(u))


def sin2pi(u: float) -> float:
    return float(lib().orc_sin2pi(u))
