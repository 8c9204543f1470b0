"""The C-ABI library builds, loads and exports every symbol include/peat.h declares (CPU only)."""
import ctypes
import math
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def declared_functions():
    text = (ROOT / "include" / "peat.h").read_text()
    return sorted(set(re.findall(r"^(?:peat_status_t|const char\*|void|int32_t|double)\s+(peat_\w+)\s*\(", text, re.M)))


def test_header_declares_the_boundary():
    assert declared_functions() == sorted([
        "peat_compare", "peat_compare_noalloc", "peat_compare_segmented", "peat_inject_compare", "peat_last_error",
        "peat_isclose_grid", "peat_mean_std", "peat_pseudo_error_inject", "peat_signature_create",
        "peat_signature_destroy",
        "peat_set_stage1_event", "peat_spearman", "peat_tensor_stats", "peat_test_for_digits",
        "peat_test_noalloc_expire_waits", "peat_test_quot_rn", "peat_topk_mean", "peat_trend"])


def test_library_builds_and_exports_every_declared_symbol():
    from paper_2609_13544_gb300 import buildlib
    lib = buildlib.build()
    L = ctypes.CDLL(str(lib))
    for name in declared_functions():
        assert hasattr(L, name), name


def test_binding_names_match_the_abi():
    import paper_2609_13544_gb300 as peat
    for name in declared_functions():
        assert hasattr(peat, name), name
    assert peat.STATS_DTYPE.itemsize == 160
    assert peat.TOPK_DTYPE.itemsize == 48
    assert peat.TSTATS_DTYPE.itemsize == 80


def test_last_error_without_handle_is_empty_string():
    import paper_2609_13544_gb300 as peat
    peat.build()
    assert isinstance(peat.peat_last_error(None), str)


def test_stats_layout_matches_oracle():
    import oracle
    import paper_2609_13544_gb300 as peat
    # the library's record is the oracle's C record followed by the Mean and
    # Variance of Errors scores, which the oracle forms from its exact sums
    # in Python (oracle.mean_var)
    assert ctypes.sizeof(oracle.Stats) + 16 == peat.STATS_DTYPE.itemsize
    assert [f for f, _ in oracle.Stats._fields_] + ["mean_abs", "var_abs"] == list(peat.STATS_DTYPE.names)


def test_digit_split_and_its_range_check():
    """The exact accumulators' digit split (run on the host through the testing
    aid): every in-range term comes back exactly as its digits (checked with
    Python integers), and a term that needs a digit outside the 24 is reported,
    never written.  The range is [2^-416, 2^352): digit j weighs 2^(32 j - 416)."""
    import random
    import paper_2609_13544_gb300 as peat
    rng = random.Random(5)
    for _ in range(2000):
        bits = rng.choice([1, 24, 53, 64, 100, 128])
        m = rng.getrandbits(bits) | 1
        e = rng.randint(-416, 352 - bits)
        neg = rng.random() < 0.5
        d, dropped = peat.peat_test_for_digits(m, e, neg)
        assert not dropped, (m, e)
        total = sum(int(v) << (32 * j) for j, v in enumerate(d))  # value * 2^416
        assert total == (-1 if neg else 1) * (m << (e + 416)), (m, e, neg)
        assert all(abs(int(v)) < 2 ** 32 for v in d)
    # the edges: the lowest digit's lowest bit, the highest digit's highest bit
    d, dropped = peat.peat_test_for_digits(1, -416, False)
    assert not dropped and int(d[0]) == 1 and not d[1:].any()
    d, dropped = peat.peat_test_for_digits(1, 351, True)
    assert not dropped and int(d[23]) == -(2 ** 31) and not d[:23].any()
    # out of range below and above: reported, and nothing of it written
    for m, e in [(1, -417), (1, 352), (3, 351), (2 ** 127 + 1, 300), (5, -1000)]:
        d, dropped = peat.peat_test_for_digits(m, e, False)
        assert dropped, (m, e)
    d, dropped = peat.peat_test_for_digits(3, 351, False)  # 2^351 kept, 2^352 reported
    assert dropped and int(d[23]) == 2 ** 31
    d, dropped = peat.peat_test_for_digits(0, 10 ** 4, False)  # zero: nothing at all
    assert not dropped and not d.any()


def _rn(q):
    from fractions import Fraction  # noqa: F401
    try:
        return float(q)
    except OverflowError:
        return math.inf


def test_quotient_rounding_of_the_mean_and_variance():
    """The one rounding of the Mean and Variance of Errors scores (run on the
    host through the testing aid): RN-even binary64 of (W + f) 2^e / d against
    Python's correctly rounded Fraction -> float, over random operands and the
    edges: exact quotients, ties to even, the subnormal grid, the overflow
    threshold, d = 1 and d = 2^64 - 1.  f = 1/2 stands for any 0 < f < 1 (the
    quotient keeps 63 bits or more, so no rounding boundary lies inside)."""
    import random
    from fractions import Fraction
    import paper_2609_13544_gb300 as peat
    rng = random.Random(11)

    def want(W, sticky, e, d):
        return _rn(Fraction(2 * W + (1 if sticky else 0), 2 * d) * Fraction(2) ** e)

    cases = []
    for _ in range(4000):
        W = (1 << 127) | rng.getrandbits(127)
        d = rng.choice([1, 2, 3, 7, 10, rng.getrandbits(16) | 1, rng.getrandbits(32) | 1, rng.getrandbits(63) | 1,
                        (1 << 64) - 1, rng.getrandbits(64) | 1])
        e = rng.choice([rng.randint(-1300, 1000), rng.randint(-1250, -1150), rng.randint(-200, 200)])
        cases.append((W, rng.random() < 0.5, e, d))
    # exact quotients on the grid and ties between grid points
    for _ in range(500):
        d = rng.getrandbits(rng.choice([8, 30, 60])) | 1
        q = ((1 << 52) | rng.getrandbits(52)) * 2 + rng.choice([0, 1])  # a grid value or a midpoint (54 bits)
        W = q * d
        sh = 128 - W.bit_length()
        cases.append((W << sh, False, rng.randint(-1200, 900) - sh, d))
        cases.append((W << sh, True, rng.randint(-1200, 900) - sh, d))
    # the overflow threshold (2^54 - 1) 2^970 and the largest double
    for d in (1, 3, (1 << 64) - 1):
        for q in ((1 << 54) - 1, (1 << 54) - 2, (1 << 53) - 1):
            W = q * d
            sh = 128 - W.bit_length()
            cases.append((W << sh, False, 970 - sh, d))
            cases.append((W << sh, True, 970 - sh, d))
    for W, sticky, e, d in cases:
        got, exp = peat.peat_test_quot_rn(W, sticky, e, d), want(W, sticky, e, d)
        assert got == exp, (hex(W), sticky, e, d, got, exp)
