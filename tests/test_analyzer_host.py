"""The Analyzer's host-side steps (Section IV-C): Spearman rank correlation
(IV-C-2) and the model-wise (mean, std) error range (IV-C-1).  The oracle is
pinned to scipy and Python's statistics module; the C library's host
functions are checked against the oracle.  No GPU work."""
import math
import statistics

import numpy as np
import pytest


def _data(seed, n, ties):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal(n)
    y = 0.6 * x + 0.8 * rng.standard_normal(n)
    if ties:
        x = np.round(x * 2) / 2
        y = np.round(y)
    return x, y


@pytest.mark.parametrize("n,ties", [(2, False), (10, True), (107, False), (400, True), (2000, True)])
def test_oracle_spearman_against_scipy(oracle, n, ties):
    stats = pytest.importorskip("scipy.stats")
    x, y = _data(n, n, ties)
    want = stats.spearmanr(x, y).statistic
    assert math.isclose(oracle.spearman(x, y), want, rel_tol=1e-12, abs_tol=1e-15)


def test_oracle_spearman_closed_forms(oracle):
    x = [0.5, 1.5, 2.0, 7.0, 9.5]
    assert oracle.spearman(x, [v * 3 - 1 for v in x]) == 1.0
    assert oracle.spearman(x, [-v for v in x]) == -1.0
    assert math.isnan(oracle.spearman(x, [2.0] * 5))
    assert math.isnan(oracle.spearman([1.0], [2.0]))
    # one tie: ranks of y are 1, 2, 3, 4.5, 4.5; centred cross sum 9.5, squares 10 and 9.5,
    # so rho = 9.5 / sqrt(10 * 9.5) = sqrt(0.95)
    rho = oracle.spearman([1, 2, 3, 4, 5], [1, 2, 3, 4, 4])
    assert math.isclose(rho, math.sqrt(0.95), rel_tol=1e-15)
    # monotone transforms do not change it
    a, b = _data(3, 300, False)
    assert oracle.spearman(a, b) == oracle.spearman(np.exp(a), b ** 3)


def test_oracle_mean_std_against_statistics(oracle):
    rng = np.random.default_rng(11)
    x = list(rng.standard_normal(400) * 1e-3 + 2.0)
    m, sd = oracle.mean_std(x, 0)
    assert m == statistics.fmean(x) or math.isclose(m, statistics.fmean(x), rel_tol=1e-16)
    assert math.isclose(sd, statistics.pstdev(x), rel_tol=1e-15)
    m1, sd1 = oracle.mean_std(x, 1)
    assert math.isclose(sd1, statistics.stdev(x), rel_tol=1e-15)
    assert oracle.mean_std([5.0], 0) == (5.0, 0.0)
    assert math.isnan(oracle.mean_std([5.0], 1)[1])


@pytest.fixture(scope="module")
def peat_host():
    import paper_2609_13544_gb300 as peat
    from paper_2609_13544_gb300 import buildlib
    buildlib.build()
    peat.load()
    return peat


@pytest.mark.parametrize("n,ties", [(2, False), (10, True), (107, False), (400, True), (5000, True)])
def test_library_spearman_matches_oracle(peat_host, oracle, n, ties):
    x, y = _data(100 + n, n, ties)
    assert math.isclose(peat_host.peat_spearman(x, y), oracle.spearman(x, y), rel_tol=1e-14, abs_tol=1e-16)


def test_library_spearman_edges(peat_host):
    assert math.isnan(peat_host.peat_spearman([1.0], [1.0]))
    assert math.isnan(peat_host.peat_spearman([1.0, 1.0, 1.0], [1.0, 2.0, 3.0]))
    assert peat_host.peat_spearman([1.0, 2.0, 3.0], [3.0, 2.0, 1.0]) == -1.0
    with pytest.raises(peat_host.PeatError):
        peat_host.peat_spearman([1.0, float("nan")], [1.0, 2.0])
    assert "finite" in peat_host.peat_last_error(None)


@pytest.mark.parametrize("ddof", [0, 1])
def test_library_mean_std_matches_oracle(peat_host, oracle, ddof):
    rng = np.random.default_rng(5 + ddof)
    for n, scale in [(1, 1.0), (2, 1.0), (400, 1e-6), (40000, 1e3)]:
        x = rng.standard_normal(n) * scale + 7.0
        m, sd = peat_host.peat_mean_std(x, ddof)
        om, osd = oracle.mean_std(x, ddof)
        assert math.isclose(m, om, rel_tol=1e-15)
        if math.isnan(osd):
            assert math.isnan(sd)
        else:
            assert math.isclose(sd, osd, rel_tol=1e-12, abs_tol=1e-300)
    with pytest.raises(peat_host.PeatError):
        peat_host.peat_mean_std([1.0], 2)


# ---------------------------------------------------------------- cross-step trend
def test_oracle_trend_against_polyfit_and_closed_forms(oracle):
    """The trend against numpy.polyfit on the logs, and exact power laws."""
    rng = np.random.default_rng(21)
    x = np.arange(1, 64, dtype=np.float64)
    y = 3e-5 * x ** 0.5 * np.exp(0.05 * rng.standard_normal(x.size))
    t = oracle.trend(x, y)
    b, a = np.polyfit(np.log(x), np.log(y), 1)
    assert math.isclose(t["slope"], b, rel_tol=1e-12) and math.isclose(t["intercept"], a, rel_tol=1e-12)
    r = np.log(y) - (a + b * np.log(x))
    assert math.isclose(t["r2"], 1 - (r @ r) / np.sum((np.log(y) - np.log(y).mean()) ** 2), rel_tol=1e-10)
    for p in (0.5, 1.0, -2.0):
        t = oracle.trend(x, 7.0 * x ** p)
        assert abs(t["slope"] - p) < 1e-13 and abs(t["intercept"] - math.log(7.0)) < 1e-12
        assert abs(t["r2"] - 1.0) < 1e-12
    # points outside the log domain are left out; too few points give NaN
    t = oracle.trend([0.0, 1.0, 2.0, 4.0, 5.0], [1.0, 2.0, 4.0, 0.0, math.inf])
    assert t["used"] == 2 and abs(t["slope"] - 1.0) < 1e-15
    assert math.isnan(oracle.trend([1.0], [1.0])["slope"])
    assert math.isnan(oracle.trend([2.0, 2.0], [1.0, 3.0])["slope"])
    assert math.isnan(oracle.trend([1.0, 2.0], [3.0, 3.0])["r2"])


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_library_trend_matches_oracle(peat_host, oracle, seed):
    rng = np.random.default_rng(seed)
    n = [2, 64, 5000][seed]
    x = np.arange(n, dtype=np.float64)  # x = 0 is left out on both sides
    y = np.abs(rng.standard_normal(n)) * (x + 1) ** 0.7
    y[rng.integers(0, n, max(1, n // 10))] = 0.0
    got, want = peat_host.peat_trend(x, y), oracle.trend(x, y)
    assert got["used"] == want["used"]
    for k in ("slope", "intercept", "r2"):
        if math.isnan(want[k]):
            assert math.isnan(got[k]), k
        else:
            assert math.isclose(got[k], want[k], rel_tol=1e-11, abs_tol=1e-13), (k, got[k], want[k])


def test_library_trend_edges(peat_host):
    t = peat_host.peat_trend([1.0, 2.0, 4.0], [3.0, 6.0, 12.0])
    assert abs(t["slope"] - 1.0) < 1e-15 and t["used"] == 3 and abs(t["r2"] - 1.0) < 1e-15
    t = peat_host.peat_trend([1.0], [1.0])
    assert t["used"] == 1 and math.isnan(t["slope"]) and math.isnan(t["r2"])
    t = peat_host.peat_trend([], [])
    assert t["used"] == 0 and math.isnan(t["intercept"])
