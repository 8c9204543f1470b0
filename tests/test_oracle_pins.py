"""Pins for the oracle against things other than itself (CPU only).

Each block names what it pins: hand-worked cases (tests/golden), brute force
over every 16-bit pattern, exact rational arithmetic on random pairs, library
routines (torch.isclose, torch.argmax, math.fsum, numpy.frexp), invariants
and closed forms of the synthetic recipes.  The definitions pinned are those
of Section IV-B-3 (error = |golden - faulty|, scored by max, mean and
variance) with the readings for the relative error, ULP distance, classes
and histogram bins recorded in the oracle's header.
"""
import json
import math
import struct
from fractions import Fraction
from pathlib import Path

import numpy as np
import pytest
import torch

GOLD = json.loads((Path(__file__).parent / "golden" / "hand_cases.json").read_text())
CLASS_IDX = {"exact": 0, "within_tol": 1, "mismatch": 2, "nan_inf_asym": 3, "sign_flip": 4}
NP_BITS = {"f32": np.uint32, "f16": np.uint16, "bf16": np.uint16, "f8e4m3": np.uint8, "f8e5m2": np.uint8,
           "f64": np.uint64}
FP8 = {"f8e4m3": "float8_e4m3fn", "f8e5m2": "float8_e5m2"}
_FP8_TABLE = {}


def fp8_table(dtype):
    """Every 8-bit pattern's value, from torch's own float8 conversions (OCP FP8)."""
    if dtype not in _FP8_TABLE:
        t = torch.arange(256, dtype=torch.int32).to(torch.uint8).view(getattr(torch, FP8[dtype]))
        _FP8_TABLE[dtype] = t.to(torch.float32).tolist()
    return _FP8_TABLE[dtype]


# ---------------------------------------------------------------- helpers
def decode(bits: int, dtype: str) -> float:
    """Exact value of one bit pattern via the platform's own float formats."""
    if dtype == "f32":
        return float(np.array([bits], np.uint32).view(np.float32)[0])
    if dtype == "f16":
        return float(np.array([bits], np.uint16).view(np.float16)[0])
    if dtype in FP8:
        return fp8_table(dtype)[bits]
    if dtype == "f64":
        return float(np.array([bits], np.uint64).view(np.float64)[0])
    return float(np.array([bits << 16], np.uint32).view(np.float32)[0])


def signbit(bits: int, dtype: str) -> int:
    return (bits >> {"f32": 31, "f8e4m3": 7, "f8e5m2": 7, "f64": 63}.get(dtype, 15)) & 1


def rn32(x: float) -> float:
    return float(np.float32(x))


def ref_pair(gb: int, cb: int, dtype: str, rtol: float, atol: float, rank=None):
    """The definitions evaluated with exact rationals (Python Fractions)."""
    gv, cv = decode(gb, dtype), decode(cb, dtype)
    out = {}
    gfin, cfin = math.isfinite(gv), math.isfinite(cv)
    if not (gfin and cfin):
        eq = (math.isnan(gv) and math.isnan(cv)) or (math.isinf(gv) and math.isinf(cv) and gv == cv)
        out["cls"] = 0 if eq else 3
        out["relbin"] = 0 if eq else 63
        out["finite"] = False
        return out
    out["finite"] = True
    d = Fraction(cv) - Fraction(gv)
    a = abs(d)
    ag = abs(Fraction(gv))
    R, A = Fraction(rn32(rtol)), Fraction(rn32(atol))
    if a == 0:
        cls = 0
    elif a <= A + R * ag:
        cls = 1
    elif gv != 0 and cv != 0 and signbit(gb, dtype) != signbit(cb, dtype):
        cls = 4
    else:
        cls = 2
    out["cls"] = cls
    if a == 0:
        out["relbin"], out["rel"] = 0, Fraction(0)
    elif ag == 0:
        out["relbin"], out["rel"] = 63, None
    else:
        rel = a / ag
        k = 0
        while Fraction(2) ** k > rel:
            k -= 1
        while Fraction(2) ** (k + 1) <= rel:
            k += 1
        out["relbin"], out["rel"] = min(max(k + 48, 1), 62), rel
    out["d"], out["a"] = d, a
    return out


def check_mean_var(st, absd):
    """The Mean and Variance of Errors scores (Section IV-B-3) against the
    statistics module run on the exact |d| values (Fractions in, Fractions
    out: statistics.fmean would round, mean and pvariance do not)."""
    import statistics
    if not absd:
        assert st["mean_abs"] == 0.0 and st["var_abs"] == 0.0
        return
    assert st["mean_abs"] == rn64(statistics.mean(absd))
    assert st["var_abs"] == rn64(statistics.pvariance(absd))


# ---------------------------------------------------------------- hand cases
@pytest.mark.parametrize("case", GOLD["cases"], ids=lambda c: f"{c['dtype']}:{c['g']}:{c['c']}:{c['why'][:20]}")
def test_hand_case(oracle, case):
    dt = case["dtype"]
    g = np.array([int(case["g"], 16)], NP_BITS[dt])
    c = np.array([int(case["c"], 16)], NP_BITS[dt])
    st, h = oracle.compare(g, c, dt, case["rtol"], case["atol"])
    assert st["count"][CLASS_IDX[case["class"]]] == 1, (case, st["count"])
    assert h[0][case["relbin"]] == 1 and h[0].sum() == 1, np.nonzero(h[0])
    assert h[1][case["ulpbin"]] == 1 and h[1].sum() == 1, np.nonzero(h[1])
    if case["u"] is None and case["class"] != "mismatch":
        assert st["argmax_ulp"] == -1
    elif case["u"] is not None:
        assert st["max_ulp"] == case["u"] and st["argmax_ulp"] == 0


@pytest.mark.parametrize("agg", GOLD["aggregates"], ids=lambda a: a["why"][:30])
def test_hand_aggregate(oracle, agg):
    npt = {"f32": np.float32, "f16": np.float16}[agg["dtype"]]
    st, h = oracle.compare(np.array(agg["g"], npt), np.array(agg["c"], npt), agg["dtype"], agg["rtol"], agg["atol"])
    assert st["count"] == agg["counts"]
    for k in ("n_finite", "max_abs", "argmax_abs", "max_rel", "argmax_rel", "max_ulp", "argmax_ulp",
              "sum_signed", "sum_abs", "sum_sq", "mean_abs", "var_abs"):
        assert st[k] == agg[k], k
    assert {str(i): int(v) for i, v in enumerate(h[0]) if v} == agg["relhist"]
    assert {str(i): int(v) for i, v in enumerate(h[1]) if v} == agg["ulphist"]


# ---------------------------------------------------------------- ULP distance, brute force
@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_ulp_key_is_rank_for_every_16bit_pattern(oracle, dtype):
    """key(x) must equal the signed rank of x among all distinct non-NaN values
    (both zeros merged).  Since u = |key(c) - key(g)|, this fixes the ULP
    distance of all 2^32 pairs of the type."""
    allbits = np.arange(65536, dtype=np.uint32)
    vals = np.array([decode(int(b), dtype) for b in allbits])
    ok = ~np.isnan(vals)
    distinct = np.unique(vals[ok])  # -0.0 == 0.0 merge
    rank = {v: i for i, v in enumerate(distinct.tolist())}
    r0 = rank[0.0]
    keys = np.array([oracle.ulp_key(int(b), dtype) for b in allbits[ok]])
    ranks = np.array([rank[v] - r0 for v in vals[ok].tolist()])
    assert np.array_equal(keys, ranks)


def test_ulp_key_f32_successor(oracle):
    rng = np.random.default_rng(1)
    bits = rng.integers(0, 2 ** 32, 20000, dtype=np.uint64).astype(np.uint32)
    bits = np.concatenate([bits, np.array([0, 0x80000000, 1, 0x80000001, 0x7f7fffff, 0xff7fffff, 0x00800000], np.uint32)])
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    x = x[x < np.float32(3.4028235e38)]
    up = np.nextafter(x, np.float32(np.inf))
    for a, b in zip(x.view(np.uint32)[:5000], up.view(np.uint32)[:5000]):
        assert oracle.ulp_key(int(b), "f32") == oracle.ulp_key(int(a), "f32") + 1
    assert oracle.ulp_key(0, "f32") == oracle.ulp_key(0x80000000, "f32") == 0


# ---------------------------------------------------------------- 8-bit types, every pair
def test_fp8_formats_against_the_specification(oracle):
    """OCP FP8: E4M3 has no infinities, its only NaNs are 0x7F / 0xFF and
    0x7E = 448 is its largest value; E5M2 is IEEE-like (0x7C = +Inf, 0x7B =
    57344); subnormal steps 2^-9 and 2^-16."""
    e4, e5 = fp8_table("f8e4m3"), fp8_table("f8e5m2")
    assert e4[0x7E] == 448.0 and math.isnan(e4[0x7F]) and math.isnan(e4[0xFF]) and e4[0x01] == 2.0 ** -9
    assert sum(math.isnan(v) for v in e4) == 2 and not any(math.isinf(v) for v in e4)
    assert e5[0x7B] == 57344.0 and e5[0x7C] == math.inf and e5[0xFC] == -math.inf and e5[0x01] == 2.0 ** -16
    assert sum(math.isnan(v) for v in e5) == 6
    # the oracle decodes the same values: compare each pattern with +0 (d = the value)
    for dt, tab in (("f8e4m3", e4), ("f8e5m2", e5)):
        c = np.arange(256, dtype=np.uint8)
        stats, _ = oracle.compare_segmented(np.zeros(256, np.uint8), c, np.arange(257), dt, 0.0, 0.0)
        for b in range(256):
            if math.isfinite(tab[b]):
                assert stats[b]["sum_signed"] == tab[b] and stats[b]["n_finite"] == 1, (dt, b)
            else:
                assert stats[b]["n_finite"] == 0 and stats[b]["count"][3] == 1, (dt, b)


@pytest.mark.parametrize("dtype", ["f8e4m3", "f8e5m2"])
@pytest.mark.parametrize("tol", [(0.0, 0.0), (0.125, 2.0 ** -7)])
def test_fp8_every_pair_against_exact_rationals(oracle, dtype, tol):
    """All 65,536 (golden, candidate) pairs of the type: class, both bins, the
    ULP distance as the distance of signed ranks among the distinct non-NaN
    values, and the exact error terms."""
    rtol, atol = tol
    tab = fp8_table(dtype)
    distinct = sorted({v for v in tab if not math.isnan(v)})
    pos = {v: i for i, v in enumerate(distinct)}
    rank = [None if math.isnan(v) else pos[v] - pos[0.0] for v in tab]
    g = np.repeat(np.arange(256, dtype=np.uint8), 256)
    c = np.tile(np.arange(256, dtype=np.uint8), 256)
    stats, hist = oracle.compare_segmented(g, c, np.arange(g.size + 1), dtype, rtol, atol)
    for i in range(g.size):
        gb, cb = int(g[i]), int(c[i])
        ref = ref_pair(gb, cb, dtype, rtol, atol)
        st = stats[i]
        assert st["count"][ref["cls"]] == 1, (hex(gb), hex(cb), ref, st["count"])
        assert hist[i][0][ref["relbin"]] == 1, (hex(gb), hex(cb), ref["relbin"])
        rg, rc = rank[gb], rank[cb]
        if rg is None or rc is None:
            assert st["argmax_ulp"] == -1 and hist[i][1][0 if (rg is None and rc is None) else 63] == 1
        else:
            assert st["max_ulp"] == abs(rc - rg) and hist[i][1][min(abs(rc - rg), 63)] == 1
        if ref["finite"]:
            assert st["sum_signed"] == float(ref["d"]) and st["sum_abs"] == float(ref["a"])
            assert st["sum_sq"] == float(ref["d"] ** 2) and st["max_abs"] == float(ref["a"])
            assert st["max_rel"] == (math.inf if ref["rel"] is None else float(ref["rel"]))


# ---------------------------------------------------------------- binary64
def rn64(q: Fraction) -> float:
    """Round-to-nearest binary64 of an exact rational, +-inf past the largest double."""
    try:
        return float(q)
    except OverflowError:  # the rounded value is past the largest double
        return math.inf if q > 0 else -math.inf


def _random_f64_pairs(n, rng):
    """Mixture: relative noise, one-ULP neighbours, arbitrary patterns, sign flips,
    zeros, subnormals, and operands near the largest double (the difference overflows)."""
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


def test_f64_ulp_key_successor(oracle):
    rng = np.random.default_rng(64)
    x = (rng.standard_normal(3000) * np.exp2(rng.integers(-1000, 1000, 3000))).astype(np.float64)
    x = np.concatenate([x, [0.0, 5e-324, -5e-324, 2.2250738585072014e-308, 1.7976931348623157e308]])
    with np.errstate(over="ignore"):  # the largest double steps to +inf, one key further
        up = np.nextafter(x, np.inf)
    for a, b in zip(x.view(np.uint64), up.view(np.uint64)):
        assert oracle.ulp_key(int(b), "f64") == oracle.ulp_key(int(a), "f64") + 1, hex(int(a))
    assert oracle.ulp_key(0, "f64") == oracle.ulp_key(1 << 63, "f64") == 0
    inf = int(np.array([np.inf]).view(np.uint64)[0])
    assert oracle.ulp_key(inf, "f64") == oracle.ulp_key(0x7FEFFFFFFFFFFFFF, "f64") + 1


def test_f64_per_pair_against_exact_rationals(oracle):
    rng = np.random.default_rng(641)
    g, c = _random_f64_pairs(2500, rng)
    rtol, atol = 1e-9, 1e-300
    stats, hist = oracle.compare_segmented(g, c, np.arange(g.size + 1), "f64", rtol, atol)
    for i in range(g.size):
        ref = ref_pair(int(g[i]), int(c[i]), "f64", rtol, atol)
        st = stats[i]
        assert st["count"][ref["cls"]] == 1, (i, hex(g[i]), hex(c[i]), ref, st["count"])
        assert hist[i][0][ref["relbin"]] == 1, (i, ref["relbin"], np.nonzero(hist[i][0]))
        if ref["finite"]:
            assert st["sum_signed"] == rn64(ref["d"]) and st["sum_abs"] == rn64(ref["a"])
            assert st["sum_sq"] == rn64(ref["d"] ** 2) and st["max_abs"] == rn64(ref["a"])
            assert st["max_rel"] == (math.inf if ref["rel"] is None else rn64(ref["rel"])), (hex(g[i]), hex(c[i]))


def test_f64_aggregate_against_exact_rationals(oracle):
    rng = np.random.default_rng(642)
    g, c = _random_f64_pairs(1500, rng)
    g[900], c[900] = g[400], c[400]  # a tie for the maxima
    st, hist = oracle.compare(g, c, "f64", 1e-6, 0.0)
    S0 = S1 = S2 = Fraction(0)
    best_a = best_r = None
    ia = ir = -1
    absd = []
    for i in range(g.size):
        ref = ref_pair(int(g[i]), int(c[i]), "f64", 1e-6, 0.0)
        if not ref["finite"]:
            continue
        absd.append(ref["a"])
        S0 += ref["d"]
        S1 += ref["a"]
        S2 += ref["d"] ** 2
        if best_a is None or ref["a"] > best_a:
            best_a, ia = ref["a"], i
        r = ref["rel"] if ref["rel"] is not None else math.inf
        if best_r is None or r > best_r:
            best_r, ir = r, i
    assert (st["sum_signed"], st["sum_abs"], st["sum_sq"]) == (rn64(S0), rn64(S1), rn64(S2))
    check_mean_var(st, absd)
    assert st["argmax_abs"] == ia and st["max_abs"] == rn64(best_a)
    assert st["argmax_rel"] == ir
    assert st["max_rel"] == (math.inf if best_r == math.inf else rn64(best_r))


def test_f64_range_edges(oracle):
    """Differences past the largest double, subnormal sums that round, and a
    quotient past the rounding threshold of the largest double."""
    big, tiny = 1.7976931348623157e308, 5e-324
    g = np.array([-big, 0.0, tiny, 2 * tiny, 1e-300], np.float64)
    c = np.array([big, 3 * tiny, 0.0, 0.0, 1e10], np.float64)
    st, _ = oracle.compare(g, c, "f64", 0.0, 0.0)
    d = [Fraction(float(b)) - Fraction(float(a)) for a, b in zip(g, c)]
    assert st["max_abs"] == math.inf and st["argmax_abs"] == 0     # 2 * big rounds past the largest double
    assert st["sum_signed"] == rn64(sum(d)) == math.inf
    assert st["sum_sq"] == rn64(sum(x * x for x in d)) == math.inf
    st, _ = oracle.compare(g[1:4], c[1:4], "f64", 0.0, 0.0)
    dd = [Fraction(float(b)) - Fraction(float(a)) for a, b in zip(g[1:4], c[1:4])]
    assert st["sum_sq"] == rn64(sum(x * x for x in dd)) == 0.0       # squares far below the smallest subnormal
    assert st["sum_abs"] == rn64(sum(abs(x) for x in dd)) == 6 * tiny
    assert st["max_rel"] == math.inf                                # g = 0 < |d|
    st, _ = oracle.compare(g[4:], c[4:], "f64", 0.0, 0.0)
    assert st["max_rel"] == math.inf                                # 1e10 / 1e-300 rounds past the largest double


# ---------------------------------------------------------------- exact rationals on random pairs
def _random_pairs(dtype, n, rng):
    w = 32 if dtype == "f32" else 16
    top = 2 ** w
    g = rng.integers(0, top, n, dtype=np.uint64)
    c = g.copy()
    kind = rng.integers(0, 6, n)
    # 0: close in key space, 1: random pattern, 2: sign flipped close, 3: zero candidate,
    # 4: same value, 5: small values near the subnormal range
    step = rng.integers(-4, 5, n)
    c = np.where(kind == 0, (g + step.astype(np.uint64)) % top, c)
    c = np.where(kind == 1, rng.integers(0, top, n, dtype=np.uint64), c)
    sign = np.uint64(1 << (w - 1))
    c = np.where(kind == 2, (g ^ sign) + (step.astype(np.uint64) % np.uint64(3)), c) % top
    c = np.where(kind == 3, np.uint64(0), c)
    small = rng.integers(0, 2 ** (w // 2), n, dtype=np.uint64)
    g = np.where(kind == 5, small, g)
    c = np.where(kind == 5, small + rng.integers(0, 3, n).astype(np.uint64), c)
    return g.astype(NP_BITS[dtype]), c.astype(NP_BITS[dtype])


_RANKS = {}


def rank_table(dtype):
    """Signed rank of every 16-bit pattern among the distinct non-NaN values."""
    if dtype not in _RANKS:
        vals = np.array([decode(b, dtype) for b in range(65536)])
        distinct = np.unique(vals[~np.isnan(vals)])
        pos = {v: i for i, v in enumerate(distinct.tolist())}
        r0 = pos[0.0]
        _RANKS[dtype] = [None if math.isnan(v) else pos[v] - r0 for v in vals.tolist()]
    return _RANKS[dtype]


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_per_pair_ulp_against_rank_distance(oracle, dtype):
    rng = np.random.default_rng({"f16": 31, "bf16": 32}[dtype])
    g, c = _random_pairs(dtype, 4000, rng)
    rank = rank_table(dtype)
    stats, hist = oracle.compare_segmented(g, c, np.arange(g.size + 1), dtype, 0.0, 0.0)
    for i in range(g.size):
        rg, rc = rank[int(g[i])], rank[int(c[i])]
        if rg is None or rc is None:
            both = rg is None and rc is None
            assert stats[i]["argmax_ulp"] == -1 and hist[i][1][0 if both else 63] == 1
        else:
            u = abs(rc - rg)
            assert stats[i]["max_ulp"] == u and stats[i]["argmax_ulp"] == 0
            assert hist[i][1][min(u, 63)] == 1


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_per_pair_against_exact_rationals(oracle, dtype):
    rng = np.random.default_rng({"f32": 11, "f16": 12, "bf16": 13}[dtype])
    g, c = _random_pairs(dtype, 3000, rng)
    rtol, atol = 1e-3, 1e-30
    off = np.arange(g.size + 1)
    stats, hist = oracle.compare_segmented(g, c, off, dtype, rtol, atol)
    for i in range(g.size):
        ref = ref_pair(int(g[i]), int(c[i]), dtype, rtol, atol)
        st = stats[i]
        assert st["count"][ref["cls"]] == 1, (i, hex(g[i]), hex(c[i]), ref, st["count"])
        assert hist[i][0][ref["relbin"]] == 1, (i, ref["relbin"], np.nonzero(hist[i][0]))
        if ref["finite"]:
            assert st["n_finite"] == 1
            assert st["sum_signed"] == float(ref["d"])
            assert st["sum_abs"] == float(ref["a"])
            assert st["sum_sq"] == float(ref["d"] ** 2)
            assert st["max_abs"] == float(ref["a"])
            exp_rel = math.inf if ref["rel"] is None else float(ref["rel"])
            assert st["max_rel"] == exp_rel
        else:
            assert st["n_finite"] == 0 and st["argmax_abs"] == -1


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_aggregate_against_exact_rationals(oracle, dtype):
    rng = np.random.default_rng({"f32": 21, "f16": 22, "bf16": 23}[dtype])
    g, c = _random_pairs(dtype, 1500, rng)
    # plant exact ties for the maxima at two indices
    g[700], c[700] = g[300], c[300]
    st, hist = oracle.compare(g, c, dtype, 1e-2, 0.0)
    S0 = S1 = S2 = Fraction(0)
    best_a = best_r = None
    ia = ir = -1
    absd = []
    for i in range(g.size):
        ref = ref_pair(int(g[i]), int(c[i]), dtype, 1e-2, 0.0)
        if not ref["finite"]:
            continue
        absd.append(ref["a"])
        S0 += ref["d"]
        S1 += ref["a"]
        S2 += ref["d"] ** 2
        if best_a is None or ref["a"] > best_a:
            best_a, ia = ref["a"], i
        r = ref["rel"] if ref["rel"] is not None else math.inf
        if best_r is None or r > best_r:
            best_r, ir = r, i
    assert st["sum_signed"] == float(S0)
    assert st["sum_abs"] == float(S1)
    assert st["sum_sq"] == float(S2)
    check_mean_var(st, absd)
    assert st["argmax_abs"] == ia and st["max_abs"] == float(best_a)
    assert st["argmax_rel"] == ir
    assert st["max_rel"] == (math.inf if best_r == math.inf else float(best_r))


def test_mean_var_cancellation_and_binary64_range(oracle):
    """The variance is formed exactly, then rounded once: a variance nine
    orders below mean^2 (where S2/n - mean^2 in doubles is off in the third
    digit), |d| past the largest double (mean +inf, variance 0 or +inf) and a
    variance on the subnormal grid, each against Fractions of the raw values."""
    import statistics
    c = (1 + np.arange(3) * 2.0 ** -23).astype(np.float32)
    st, _ = oracle.compare(np.zeros(3, np.float32), c, "f32", 0.0)
    vals = [Fraction(float(x)) for x in c]
    assert st["mean_abs"] == float(statistics.mean(vals))
    assert st["var_abs"] == float(statistics.pvariance(vals)) > 0
    assert st["sum_sq"] / 3 - (st["sum_abs"] / 3) ** 2 != st["var_abs"]  # the naive formula is off
    big = np.finfo(np.float64).max
    st, _ = oracle.compare(np.array([-big, -big]), np.array([big, big]), "f64", 0.0)
    assert st["mean_abs"] == math.inf and st["var_abs"] == 0.0
    st, _ = oracle.compare(np.array([-big, 0.0]), np.array([big, 0.0]), "f64", 0.0)
    assert st["mean_abs"] == big and st["var_abs"] == math.inf
    d = [3 * 2.0 ** -520, 0.0, 2.0 ** -520]
    st, _ = oracle.compare(np.zeros(3), np.array(d), "f64", 0.0)
    var = statistics.pvariance([Fraction(x) for x in d])
    assert 0 < st["var_abs"] < 2.0 ** -1022 and st["var_abs"] == float(var)
    # non-finite pairs are left out of both scores
    st, _ = oracle.compare(np.array([0.0, 0.0, 1.0], np.float32), np.array([2.0, np.nan, np.inf], np.float32),
                           "f32", 0.0)
    assert st["n_finite"] == 1 and st["mean_abs"] == 2.0 and st["var_abs"] == 0.0


def test_playback_sweep_against_its_closed_form(oracle):
    """Config 5's recipe at a small size.  Step 0 compares every snapshot with
    itself: all EXACT.  At step s the candidate is the bf16 rounding of
    g (1 + 1e-4 sqrt(s) z), z ~ N(0, 1), for a bf16 golden g, so it differs
    from g exactly when the noise carries g out of g's own rounding interval:
    above by more than half the step up, below by more than half the step
    down (a quarter of the step at a power of two).  The expected number of
    non-EXACT pairs is the sum of those two Gaussian tails over the pairs
    (scipy.special.erfc); the oracle's count lies within 5 standard
    deviations of it.  (So the measured error does not grow like sqrt(s): the
    noise stays below half a bf16 step for small s, and the count follows the
    tail beyond it.)"""
    from scipy.special import erfc
    from paper_2609_13544_gb300 import workloads as W
    sweep = W.PlaybackSweep(n=262_144, device="cpu")
    st, _ = oracle.compare(sweep.workload(0).golden, sweep.workload(0).candidate, "bf16", 2.0 ** -7)
    assert st["exact"] == st["n"] == 262_144 and st["mean_abs"] == 0.0
    for s in (16, 32, 48, 63):
        w = sweep.workload(s)
        st, _ = oracle.compare(w.golden, w.candidate, "bf16", w.rtol)
        gb = w.golden.view(torch.int16).numpy().view(np.uint16).astype(np.uint32)
        ef, mant = (gb >> 7) & 0xFF, gb & 0x7F
        g = np.abs((gb << 16).view(np.float32).astype(np.float64))
        ok = (ef > 0) & (ef < 255)  # normal goldens (zero stays zero; none is subnormal here)
        step_up = np.exp2(ef.astype(np.float64) - 127 - 7)
        step_dn = np.where(mant == 0, step_up / 2, step_up)
        sig = 1e-4 * np.sqrt(s)
        p = 0.5 * (erfc(step_up / 2 / g / sig / np.sqrt(2)) + erfc(step_dn / 2 / g / sig / np.sqrt(2)))
        p = np.where(ok, p, 0.0)
        mu, sd = p.sum(), np.sqrt((p * (1 - p)).sum())
        assert abs((st["n"] - st["exact"]) - mu) <= 5 * sd + 1, (s, st["n"] - st["exact"], mu, sd)


# ---------------------------------------------------------------- library routines
def _fp16_noise(n, seed, frac_nan=0.0):
    rng = np.random.default_rng(seed)
    g = (rng.laplace(0, 0.02, n)).astype(np.float16)
    c = (g.astype(np.float32) * (1 + 1e-3 * rng.standard_normal(n).astype(np.float32))).astype(np.float16)
    if frac_nan:
        idx = rng.choice(n, int(n * frac_nan), replace=False)
        c[idx] = np.float16(np.nan)
    return g, c


def test_isclose_count_matches_exact_plus_within(oracle):
    """torch.isclose(c, g, rtol, atol, equal_nan=True) evaluated in float64 is
    exact for fp16 data with atol = 0, so its count is EXACT + WITHIN_TOL."""
    g, c = _fp16_noise(50000, 5, frac_nan=0.001)
    g[:10] = np.float16(np.inf)
    c[:5] = np.float16(np.inf)
    st, _ = oracle.compare(g, c, "f16", 1e-3, 0.0)
    close = torch.isclose(torch.from_numpy(c.astype(np.float64)), torch.from_numpy(g.astype(np.float64)),
                          rtol=st["rtol_eff"], atol=0.0, equal_nan=True)
    assert int(close.sum()) == st["exact"] + st["within_tol"]


def test_argmax_and_fsum(oracle):
    g, c = _fp16_noise(40000, 6)
    c[123] = g[77]  # a large error somewhere
    st, _ = oracle.compare(g, c, "f16", 1e-3, 0.0)
    d = c.astype(np.float64) - g.astype(np.float64)  # exact for fp16 operands
    assert st["argmax_abs"] == int(torch.argmax(torch.from_numpy(np.abs(d))))
    assert st["max_abs"] == float(np.max(np.abs(d)))
    assert st["sum_signed"] == math.fsum(d.tolist())
    assert st["sum_abs"] == math.fsum(np.abs(d).tolist())
    sq = d * d
    assert np.all(np.abs(d[d != 0]) < 2.0 ** 12 * np.abs(d[d != 0]).min() * 2 ** 14)  # d*d exact in float64
    assert st["sum_sq"] == math.fsum(sq.tolist())


def test_rel_bin_against_frexp(oracle):
    g, c = _fp16_noise(30000, 7)
    _, h = oracle.compare(g, c, "f16", 1e-3, 0.0)
    gd, cd = g.astype(np.float64), c.astype(np.float64)
    a, ag = np.abs(cd - gd), np.abs(gd)
    bins = np.zeros(64, np.int64)
    ma, ea = np.frexp(a)
    mg, eg = np.frexp(ag)
    k = ea - eg - (ma < mg)
    sel = (a > 0) & (ag > 0)
    np.add.at(bins, np.clip(k[sel] + 48, 1, 62), 1)
    bins[0] = int((a == 0).sum())
    bins[63] = int(((a > 0) & (ag == 0)).sum())
    assert np.array_equal(h[0].astype(np.int64), bins)


def test_exact_accumulator_against_python_integers(oracle):
    rng = np.random.default_rng(8)
    for trial in range(40):
        n = int(rng.integers(1, 60))
        e = rng.integers(-300, 300, n)
        x = rng.standard_normal(n) * np.exp2(e)
        if trial % 4 == 0:  # heavy cancellation
            x = np.concatenate([x, -x[:-1]])
        y = rng.standard_normal(x.size) * np.exp2(rng.integers(-200, 200, x.size))
        assert oracle.exact_sum(x) == float(sum(Fraction(v) for v in x))
        assert oracle.exact_dot(x, y) == float(sum(Fraction(a) * Fraction(b) for a, b in zip(x, y)))
    # round-half-even at a tie and just above it
    assert oracle.exact_sum([1.0, 2.0 ** -53]) == 1.0
    assert oracle.exact_sum([1.0, 2.0 ** -53, 2.0 ** -300]) == 1.0 + 2.0 ** -52
    assert oracle.exact_sum([1.0 + 2.0 ** -52, 2.0 ** -53]) == 1.0 + 2.0 ** -51


# ---------------------------------------------------------------- invariants
@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_self_compare(oracle, dtype):
    rng = np.random.default_rng(9)
    x, _ = _random_pairs(dtype, 4000, rng)
    st, h = oracle.compare(x, x, dtype, 0.0, 0.0)
    n = x.size
    assert st["exact"] == n and sum(st["count"]) == n
    assert h[0][0] == n and h[1][0] == n
    assert st["sum_abs"] == st["sum_sq"] == st["sum_signed"] == 0.0
    vals = np.array([decode(int(b), dtype) for b in x])
    fin = np.nonzero(np.isfinite(vals))[0]
    assert st["argmax_abs"] == (fin[0] if fin.size else -1)
    assert st["argmax_rel"] == st["argmax_abs"]


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_swap_and_concatenation(oracle, dtype):
    rng = np.random.default_rng(10)
    g, c = _random_pairs(dtype, 5000, rng)
    s1, h1 = oracle.compare(g, c, dtype, 0.0, 0.0)
    s2, h2 = oracle.compare(c, g, dtype, 0.0, 0.0)
    for k in ("exact", "nan_inf_asym", "sign_flip", "n_finite"):
        assert s1[k] == s2[k]
    assert np.array_equal(h1[1], h2[1])
    assert s1["max_ulp"] == s2["max_ulp"] and s1["argmax_ulp"] == s2["argmax_ulp"]
    assert s1["sum_abs"] == s2["sum_abs"] and s1["sum_sq"] == s2["sum_sq"]
    assert s1["sum_signed"] == -s2["sum_signed"]
    assert s1["max_abs"] == s2["max_abs"] and s1["argmax_abs"] == s2["argmax_abs"]
    assert sum(s1["count"]) == g.size and h1[0].sum() == g.size and h1[1].sum() == g.size
    off = np.array([0, 0, 17, 17, 1000, 1001, 4096, 5000])
    ss, hs = oracle.compare_segmented(g, c, off, dtype, 0.0, 0.0)
    assert np.array_equal(hs.sum(axis=0), h1)
    assert [sum(s["count"][j] for s in ss) for j in range(5)] == s1["count"]
    assert ss[0]["n"] == 0 and ss[0]["argmax_abs"] == -1
    assert max(s["max_ulp"] for s in ss) == s1["max_ulp"]


# ---------------------------------------------------------------- closed forms of the recipes
def test_closed_form_bf16_rne_vs_rtz(oracle):
    """RNE and RTZ roundings of the same float32 differ by one bf16 step, so
    every differing pair has u = 1 and rel in [2^-8, 2^-7) (bin 40), and is
    within rtol = 2^-7."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c2_bf16_rne_vs_rtz(numel=1 << 18, seed=2)
    st, h = oracle.compare(w.golden, w.candidate, "bf16", 2.0 ** -7)
    differ = int((w.golden.view(torch.int16) != w.candidate.view(torch.int16)).sum())
    assert set(np.nonzero(h[0])[0]) == {0, 40}
    assert set(np.nonzero(h[1])[0]) == {0, 1}
    assert h[0][40] == differ == h[1][1]
    assert st["within_tol"] == differ and st["mismatch"] == st["sign_flip"] == st["nan_inf_asym"] == 0
    n = w.n
    assert abs(differ - n / 2) < 5 * math.sqrt(n) / 2


def test_closed_form_relative_bias(oracle):
    """c = g + 1e-4|g| puts every nonzero relative error in [2^-14, 2^-13)."""
    from paper_2609_13544_gb300 import workloads as W
    shapes = W.resnet50_param_shapes()[:12]
    w = W.c3_resnet50(seed=3, shapes=shapes)
    stats, h = oracle.compare_segmented(w.golden, w.candidate, w.offsets, "f32", 1e-5)
    for s in range(0, len(shapes), 2):
        assert set(np.nonzero(h[s][0])[0]) <= {0, 34}
        assert stats[s]["sum_signed"] > 0
        gseg = w.golden[w.offsets[s]:w.offsets[s + 1]].double()
        assert abs(stats[s]["sum_signed"] / (1e-4 * float(gseg.abs().sum())) - 1) < 1e-3


def test_closed_form_gaussian_noise_moments(oracle):
    """c = g(1+e), e ~ N(0, 1e-6): E[sum d^2] = n E[g^2] 1e-12 and
    E[sum |d|] = n E|g| sqrt(2/pi) 1e-6, up to float32 rounding of c."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c1_single_fp32(n=1 << 16, seed=0, flips=0)
    st, _ = oracle.compare(w.golden, w.candidate, "f32", 1e-5)
    g = w.golden.double()
    n = w.n
    exp_sq = float((g * g).sum()) * 1e-12
    exp_abs = float(g.abs().sum()) * math.sqrt(2 / math.pi) * 1e-6
    assert abs(st["sum_sq"] / exp_sq - 1) < 0.05
    assert abs(st["sum_abs"] / exp_abs - 1) < 0.05
    assert st["mismatch"] + st["sign_flip"] + st["nan_inf_asym"] == 0


# ---------------------------------------------------------------- injector building blocks
def test_philox_known_answers(oracle):
    """Known-answer vectors published with Philox4x32-10 (Random123)."""
    assert oracle.philox([0, 0, 0, 0], [0, 0]) == [0x6627E8D5, 0xE169C58D, 0xBC57AC4C, 0x9B00DBD8]
    assert oracle.philox([0xFFFFFFFF] * 4, [0xFFFFFFFF] * 2) == [0x408F276D, 0x41C83B0E, 0xA20BC7C6, 0x6D5451FD]
    assert oracle.philox([0x243F6A88, 0x85A308D3, 0x13198A2E, 0x03707344], [0xA4093822, 0x299F31D0]) == \
        [0xD16CFE09, 0x94FDCCEB, 0x5001E420, 0x24126EA1]


def test_logf_and_cos2pi_against_libm(oracle):
    xs = np.concatenate([np.arange(1, 1 << 24, 4099, dtype=np.float64) * 2.0 ** -24, [1.0, 0.5, 2.0 ** -24]])
    for x in xs:
        x32 = rn32(x)
        ref = math.log(x32)
        assert abs(oracle.logf(x32) - ref) <= 3e-7 * max(1.0, abs(ref)), x32
    for u in np.arange(0, 1 << 24, 3001) * 2.0 ** -24:
        assert abs(oracle.cos2pi(float(u)) - math.cos(2 * math.pi * u)) < 4e-7, u
        assert abs(oracle.sin2pi(float(u)) - math.sin(2 * math.pi * u)) < 4e-7, u
    # the quadrant boundaries, where the reduction swaps cos and sin
    for u, c, s_ in ((0.0, 1.0, 0.0), (0.25, 0.0, 1.0), (0.5, -1.0, 0.0), (0.75, 0.0, -1.0)):
        assert abs(oracle.cos2pi(u) - c) < 1e-7 and abs(oracle.sin2pi(u) - s_) < 1e-7, u


def test_box_muller_pair_moments(oracle):
    """Both components of a Box-Muller pair are N(0, 1) and independent: the
    squared radius z0^2 + z1^2 is exponential with mean 2 (P(> 2) = 1/e)."""
    n = 100000
    w = [oracle.philox([i, 0, 7, 1], [5, 0]) for i in range(n)]
    zz = np.array([oracle.normal_pair_from_words(a[0], a[1]) for a in w])
    for z in (zz[:, 0], zz[:, 1]):
        assert abs(z.mean()) < 5 / math.sqrt(n)
        assert abs(z.var() - 1) < 5 * math.sqrt(2 / n)
        kurt = ((z - z.mean()) ** 4).mean() / z.var() ** 2
        assert abs(kurt - 3) < 5 * math.sqrt(24 / n)
        assert abs((np.abs(z) < 1).mean() - 0.6826894921) < 5 * math.sqrt(0.22 / n)
    r2 = zz[:, 0].astype(np.float64) ** 2 + zz[:, 1].astype(np.float64) ** 2
    assert abs(r2.mean() - 2) < 5 * 2 / math.sqrt(n)
    assert abs((r2 > 2).mean() - math.exp(-1)) < 5 * math.sqrt(0.24 / n)
    assert abs(np.corrcoef(zz[:, 0], zz[:, 1])[0, 1]) < 5 / math.sqrt(n)
    assert abs(np.corrcoef(zz[:, 0] ** 2, zz[:, 1] ** 2)[0, 1]) < 5 / math.sqrt(n)


def test_inject_draw_blocks_are_independent(oracle):
    """One draw serves four neighbouring elements: every position in the
    block still fires at the model's rate, independently of its neighbours,
    and the noise of neighbours is independent N(0, 1) (the Box-Muller pair
    of positions 2k, 2k+1 has squared radius of mean 2, P(> 2) = 1/e)."""
    n = 400000
    src = np.full(n, 1.0, np.float32)
    rate = 0.1
    dst, cnt = oracle.inject(src, "f32", [oracle.model("signflip", x=rate)], seed=3)
    f = (dst != src.view(np.uint32)).reshape(-1, 4)
    for j in range(4):
        assert abs(f[:, j].mean() - rate) < 5 * math.sqrt(rate * (1 - rate) / (n // 4)), j
    for a, b in ((0, 1), (1, 2), (2, 3), (0, 3)):
        both = (f[:, a] & f[:, b]).mean()
        assert abs(both - rate * rate) < 5 * math.sqrt(rate * rate / (n // 4)), (a, b)
    # NaN / +Inf / -Inf in the shares 1/2, 1/4, 1/4
    dst, cnt = oracle.inject(src, "f32", [oracle.model("nan_inf", x=0.05)], seed=4)
    v = dst.view(np.float32)
    k = int(cnt[0])
    for share, hit in ((0.5, np.isnan(v)), (0.25, v == np.inf), (0.25, v == -np.inf)):
        assert abs(hit.sum() / k - share) < 5 * math.sqrt(share * (1 - share) / k)
    sigma = 2.0 ** -10
    dst, _ = oracle.inject(src, "f32", [oracle.model("add_gauss", x=sigma)], seed=5)
    e = ((dst.view(np.float32).astype(np.float64) - 1.0) / sigma).reshape(-1, 4)
    for j in range(4):
        assert abs(e[:, j].mean()) < 5 / math.sqrt(n // 4) and abs(e[:, j].var() - 1) < 0.03, j
    for a, b in ((0, 1), (2, 3)):
        r2 = e[:, a] ** 2 + e[:, b] ** 2
        assert abs(r2.mean() - 2) < 0.06 and abs((r2 > 2).mean() - math.exp(-1)) < 0.01
    for a, b in ((0, 1), (1, 2), (0, 2), (2, 3)):
        assert abs(np.corrcoef(e[:, a], e[:, b])[0, 1]) < 0.01, (a, b)
        assert abs(np.corrcoef(e[:, a] ** 2, e[:, b] ** 2)[0, 1]) < 0.015, (a, b)


def test_inject_fixed_count_models(oracle):
    rng = np.random.default_rng(12)
    src = rng.standard_normal(5000).astype(np.float32)
    models = [oracle.model("rz", k=3), oracle.model("rv", k=5), oracle.model("bitflip", k=16, bit_lo=0, bit_hi=31)]
    for m in models:
        dst, cnt = oracle.inject(src, "f32", [m], seed=42)
        diff = np.nonzero(dst != src.view(np.uint32))[0]
        assert cnt[0] == m["k"] and diff.size <= m["k"]
        if m["kind"] == "rz":
            assert diff.size == 3 and np.all(dst[diff] == 0)
        if m["kind"] == "rv":
            assert all(dst[i] in set(src.view(np.uint32).tolist()) for i in diff)
        if m["kind"] == "bitflip":
            assert diff.size == 16
            x = dst[diff] ^ src.view(np.uint32)[diff]
            assert all(bin(int(v)).count("1") == 1 for v in x)
    dst2, _ = oracle.inject(src, "f32", models, seed=42)
    dst3, _ = oracle.inject(src, "f32", models, seed=42)
    assert np.array_equal(dst2, dst3)


def test_inject_rate_and_noise_models(oracle):
    rng = np.random.default_rng(13)
    n = 200000
    src = rng.standard_normal(n).astype(np.float32)
    dst, cnt = oracle.inject(src, "f32", [oracle.model("nan_inf", x=1e-3)], seed=1)
    v = dst.view(np.float32)
    assert abs(int(cnt[0]) - n * 1e-3) < 5 * math.sqrt(n * 1e-3)
    assert int(np.isnan(v).sum() + np.isinf(v).sum()) == cnt[0]
    dst, cnt = oracle.inject(src, "f32", [oracle.model("rel_gauss", x=1e-3)], seed=2)
    e = (dst.view(np.float32).astype(np.float64) / src - 1) / 1e-3
    assert cnt[0] == n and abs(e.mean()) < 5 / math.sqrt(n) and abs(e.std() - 1) < 0.01
    dst, _ = oracle.inject(src, "f32", [oracle.model("cast_f16_rne")], seed=0)
    assert np.array_equal(dst.view(np.float32), src.astype(np.float16).astype(np.float32))
    dst, _ = oracle.inject(src, "f32", [oracle.model("cast_bf16_rne")], seed=0)
    ref = torch.from_numpy(src).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(dst.view(np.float32), ref)
    dst, _ = oracle.inject(src, "f32", [oracle.model("cast_bf16_rtz")], seed=0)
    assert np.array_equal(dst, src.view(np.uint32) & np.uint32(0xFFFF0000))
    dst, _ = oracle.inject(src, "f32", [oracle.model("cast_f16_rtz")], seed=0)
    y = dst.view(np.float32).astype(np.float16)
    up = np.nextafter(y, np.where(src >= 0, np.float16(np.inf), np.float16(-np.inf)))
    assert np.all(np.abs(y.astype(np.float64)) <= np.abs(src)) and np.all(np.abs(up.astype(np.float64)) > np.abs(src))


# ---------------------------------------------------------------- mean of the top errors
def ref_topk(g, c, dtype, num, den):
    """Mean of the top errors from exact rationals: sort every finite |c - g|,
    take the ceil(n_finite * num / den) largest, add and divide exactly."""
    a = []
    for gb, cb in zip(g.tolist(), c.tolist()):
        gv, cv = decode(int(gb), dtype), decode(int(cb), dtype)
        if math.isfinite(gv) and math.isfinite(cv):
            a.append(abs(Fraction(cv) - Fraction(gv)))
    a.sort(reverse=True)
    k = -(-len(a) * num // den)
    if k == 0:
        return {"n_finite": len(a), "k": 0, "threshold": 0.0, "sum": 0.0, "mean": 0.0}
    S = sum(a[:k], Fraction(0))
    return {"n_finite": len(a), "k": k, "threshold": float(a[k - 1]), "sum": float(S), "mean": float(S / k)}


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("frac", [(1, 10), (1, 1), (3, 7), (1, 1000)])
def test_topk_against_exact_rationals(oracle, dtype, frac):
    rng = np.random.default_rng({"f32": 31, "f16": 32, "bf16": 33}[dtype] + frac[1])
    g, c = _random_pairs(dtype, 2000, rng)
    got = oracle.topk_mean(g, c, dtype, *frac)
    assert got == ref_topk(g, c, dtype, *frac)


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_topk_whole_population_is_the_mean_error(oracle, dtype):
    # num = den takes every finite pair: the sum is the signature's sum |d|
    rng = np.random.default_rng(41)
    g, c = _random_pairs(dtype, 3000, rng)
    st, _ = oracle.compare(g, c, dtype, 1e-3, 0.0)
    got = oracle.topk_mean(g, c, dtype, 1, 1)
    assert got["k"] == got["n_finite"] == st["n_finite"]
    assert got["sum"] == st["sum_abs"]


def test_topk_ties_zeros_and_arguments(oracle):
    x = np.full(1000, 0x3F80, np.uint16)            # bf16 1.0
    y = np.full(1000, 0x3F81, np.uint16)            # one step above: every |d| = 2^-7
    got = oracle.topk_mean(x, y, "bf16", 1, 10)
    assert got == {"n_finite": 1000, "k": 100, "threshold": 2.0 ** -7, "sum": 100 * 2.0 ** -7, "mean": 2.0 ** -7}
    assert oracle.topk_mean(x, x, "bf16", 1, 10)["mean"] == 0.0      # self-compare
    nan = np.full(10, 0x7FC0, np.uint16)
    assert oracle.topk_mean(nan, nan, "bf16", 1, 10)["k"] == 0       # no finite pair
    for num, den in ((0, 10), (11, 10), (1, 0)):
        with pytest.raises(ValueError):
            oracle.topk_mean(x, y, "bf16", num, den)


# ---------------------------------------------------------------------------
# context statistics (Section IV-C-2): pinned to exact rational arithmetic on
# the decoded values and to Python's statistics module
# ---------------------------------------------------------------------------
def _decoded(bits, dtype):
    import torch
    tdt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[dtype]
    iv = torch.int32 if dtype == "f32" else torch.int16
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int32 if dtype == "f32" else np.int16)).view(tdt)
    return [float(v) for v in t.to(torch.float64).tolist()]


def ref_tstats(vals):
    from fractions import Fraction
    fin = [v for v in vals if math.isfinite(v)]
    nf = len(fin)
    s1 = sum(Fraction(v) for v in fin)
    s2 = sum(Fraction(v) * Fraction(v) for v in fin)
    out = {"n": len(vals), "n_finite": nf, "n_nan": sum(1 for v in vals if math.isnan(v)),
           "n_inf": sum(1 for v in vals if math.isinf(v)), "sum": float(s1), "sum_sq": float(s2),
           "mean": float(s1 / nf) if nf else 0.0, "var": float(s2 / nf - (s1 / nf) ** 2) if nf else 0.0}
    if nf:
        key = lambda v: (v, math.copysign(1.0, v))  # -0 below +0
        out["min"], out["max"] = min(fin, key=key), max(fin, key=key)
    else:
        out["min"] = out["max"] = 0.0
    return out


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_tensor_stats_against_exact_rationals(oracle, dtype):
    from parity_util import random_pairs
    for seed, n in [(1, 0), (2, 1), (3, 17), (4, 3000)]:
        g, c = random_pairs(dtype, n, seed)
        bits = np.concatenate([g, c])
        got = oracle.tensor_stats(bits, dtype)
        want = ref_tstats(_decoded(bits, dtype))
        for k, v in want.items():
            a = got[k]
            assert a == v and (not isinstance(v, float) or math.copysign(1, a) == math.copysign(1, v)), \
                (dtype, seed, k, a, v)


def test_tensor_stats_closed_forms(oracle):
    import statistics
    # a constant tensor has variance exactly 0; two values a, b have (a - b)^2 / 4
    c = np.full(1000, 0.1, np.float32).view(np.uint32)
    r = oracle.tensor_stats(c, "f32")
    assert r["var"] == 0.0 and r["mean"] == float(np.float32(0.1))
    ab = np.array([3.0, -1.0] * 50, np.float32).view(np.uint32)
    assert oracle.tensor_stats(ab, "f32")["var"] == 4.0
    # statistics.pvariance / fmean work in exact fractions on these doubles
    rng = np.random.default_rng(9)
    x = (rng.standard_normal(5000) * 3 + 100).astype(np.float32)
    r = oracle.tensor_stats(x.view(np.uint32), "f32")
    assert r["var"] == statistics.pvariance([float(v) for v in x])
    assert r["mean"] == statistics.mean([float(v) for v in x])
    # -0 sorts below +0 in min/max
    z = np.array([0.0, -0.0, 0.0], np.float32).view(np.uint32)
    rz = oracle.tensor_stats(z, "f32")
    assert math.copysign(1, rz["min"]) < 0 and math.copysign(1, rz["max"]) > 0
