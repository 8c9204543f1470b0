"""GPU parity on the five synthetic recipes (paper_2609_13544_gb300.workloads).

Oracle-sized cases compare every output; full-size cases, in the launch
configuration the bench times, compare the outputs the oracle can compute one
by one (whole small segments) and check properties that hold at any size.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch

from parity_util import assert_hist_equal, assert_stats_equal, oracle_segmented

pytestmark = pytest.mark.gpu

ITYPE = {"f32": torch.int32, "f16": torch.int16, "bf16": torch.int16}
NPT = {"f32": np.uint32, "f16": np.uint16, "bf16": np.uint16}


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0, max_segments=4096)
    yield handle
    handle.close()


def host_bits(t, dtype):
    return t.contiguous().view(ITYPE[dtype]).cpu().numpy().view(NPT[dtype])


def value_at(bits, i, dtype):
    """The value of element i (a Python float, exact for every format here)."""
    b = int(bits[i])
    if dtype == "f32":
        return float(np.array([b], np.uint32).view(np.float32)[0])
    if dtype == "f16":
        return float(np.array([b], np.uint16).view(np.float16)[0])
    return float(np.array([b << 16], np.uint32).view(np.float32)[0])  # bf16


def compare_workload(peat, oracle, h, w, ctx):
    gb, cb = host_bits(w.golden, w.dtype), host_bits(w.candidate, w.dtype)
    g, c = w.golden.cuda(), w.candidate.cuda()
    if w.offsets is None:
        gs, gh = peat.peat_compare(h, g, c, w.rtol, w.atol)
        os_, oh = oracle.compare(gb, cb, w.dtype, w.rtol, w.atol)
        assert_stats_equal(gs, os_, ctx)
        assert_hist_equal(gh, oh, ctx)
        return gs
    gs, gh = peat.peat_compare_segmented(h, g, c, w.offsets, w.rtol, w.atol)
    os_, oh = oracle_segmented(gb, cb, w.offsets, w.dtype, w.rtol, w.atol)
    for s in range(len(os_)):
        assert_stats_equal(gs[s], os_[s], f"{ctx} seg {s}")
    assert_hist_equal(gh, oh, ctx)
    return gs


def test_c1_single_fp32_full(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c1_single_fp32(device="cuda")
    st = compare_workload(peat_gpu, oracle, h, w, "c1")
    assert st["n"] == 1 << 20


def test_c2_bf16_reduced(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c2_bf16_rne_vs_rtz(numel=(1 << 21) + 5, device="cuda")
    compare_workload(peat_gpu, oracle, h, w, "c2-reduced")


def test_c3_resnet50_full(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c3_resnet50(device="cuda")
    st = compare_workload(peat_gpu, oracle, h, w, "c3")
    assert len(st) == 161


def test_c3_resnet50_flattened_one_segment(peat_gpu, oracle, h):
    """All 161 parameter tensors as one flat buffer: the error statistics change
    from tensor to tensor inside every CTA's range, so warps move their windows
    (and CTAs holding many general pairs rescan with the logged windows)."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c3_resnet50(device="cuda")
    w.offsets = None
    st = compare_workload(peat_gpu, oracle, h, w, "c3-flat")
    assert st["n"] == 25_557_032


def small_gpt_shapes():
    d, vocab, layers = 256, 4000, 3
    shapes = [(vocab, d), (512, d)]
    for _ in range(layers):
        shapes += [(d,), (d,), (d, 3 * d), (3 * d,), (d, d), (d,), (d,), (d,), (d, 4 * d), (4 * d,), (4 * d, d), (d,)]
    return shapes + [(d,), (d,)]


def test_c4_gpt2_like_reduced(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.c4_gpt2_medium(device="cuda", shapes=small_gpt_shapes(), nan_rate=1e-4, flip_rate=1e-4)
    st = compare_workload(peat_gpu, oracle, h, w, "c4-reduced")
    assert sum(s["nan_inf_asym"] for s in st) == len(w.meta["nan_inf_positions"])


@pytest.mark.parametrize("step", [0, 1, 63])
def test_c5_playback_reduced(peat_gpu, oracle, h, step):
    from paper_2609_13544_gb300 import workloads as W
    sweep = W.PlaybackSweep(n=(1 << 20) + 11, device="cuda")
    w = sweep.workload(step)
    st = compare_workload(peat_gpu, oracle, h, w, f"c5 step {step}")
    if step == 0:
        assert st["exact"] == w.n


def test_c5_sweep_step_by_step_and_trend(peat_gpu, oracle, h):
    """Config 5 as a sweep (Alg. 1's Err step once per recorded epoch): eight
    steps spanning 0..63 of a 1,048,576-element bf16 sweep, each compared on
    the device and by the oracle (every output bit for bit); the library's
    cross-step trend of the device's mean |d| series equals the oracle's
    trend of its own series."""
    from paper_2609_13544_gb300 import workloads as W
    sweep = W.PlaybackSweep(n=1 << 20, device="cuda")
    steps = [0, 9, 18, 27, 36, 45, 54, 63]
    dev_mean, orc_mean = [], []
    for s in steps:
        w = sweep.workload(s)
        st = compare_workload(peat_gpu, oracle, h, w, f"c5 sweep step {s}")
        if s == 0:
            assert st["exact"] == w.n
        dev_mean.append(st["mean_abs"])
        gb, cb = host_bits(w.golden, "bf16"), host_bits(w.candidate, "bf16")
        orc_mean.append(oracle.compare(gb, cb, "bf16", w.rtol, w.atol)[0]["mean_abs"])
    assert dev_mean == orc_mean
    got, want = peat_gpu.peat_trend(steps, dev_mean), oracle.trend(steps, orc_mean)
    assert got["used"] == want["used"] >= 2
    for k in ("slope", "intercept", "r2"):
        assert math.isclose(got[k], want[k], rel_tol=1e-11), k


def test_c5_sweep_resumes_from_its_records(peat_gpu, h, tmp_path):
    """The sweep driver on the CUDA path: four steps recorded, a rerun reads
    them back (no compare launched) with the same signatures, and a step
    whose record is removed is compared again and comes out the same."""
    from paper_2609_13544_gb300 import workloads as W
    from paper_2609_13544_gb300.sweep import playback_sweep
    sweep = W.PlaybackSweep(n=1 << 20, device="cuda")
    steps = [0, 21, 42, 63]
    r1 = playback_sweep(h, sweep.step, steps, 2.0 ** -7, record_dir=tmp_path, tag="c5-1M")
    assert r1["computed"] == 4 and r1["records"][0]["stats"]["exact"] == 1 << 20
    r2 = playback_sweep(h, lambda s: (_ for _ in ()).throw(AssertionError("recomputed")), steps, 2.0 ** -7,
                        record_dir=tmp_path, tag="c5-1M")
    assert r2["resumed"] == 4 and r2["series"] == r1["series"]
    (tmp_path / "step_000042.json").unlink()
    r3 = playback_sweep(h, sweep.step, steps, 2.0 ** -7, record_dir=tmp_path, tag="c5-1M")
    assert r3["computed"] == 1 and r3["series"] == r1["series"]
    assert r3["records"][2]["hist"] == r1["records"][2]["hist"]


def _check_properties(st, hist, n):
    assert sum(st["count"]) == n == st["n"]
    assert int(hist[0].sum()) == n and int(hist[1].sum()) == n
    assert int(hist[0][0]) == st["exact"] == int(hist[1][0])
    assert st["n_finite"] <= n


def test_c2_full_size_properties(peat_gpu, h):
    """[8,2048,4096] bf16 RNE vs RTZ: every differing pair is one step apart with
    rel in [2^-8, 2^-7), within rtol = 2^-7."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c2_bf16_rne_vs_rtz(device="cuda")
    st, hist = peat_gpu.peat_compare(h, w.golden, w.candidate, w.rtol, w.atol)
    _check_properties(st, hist, w.n)
    differ = int((w.golden.view(torch.int16) != w.candidate.view(torch.int16)).sum())
    assert set(np.nonzero(hist[0])[0]) <= {0, 40} and set(np.nonzero(hist[1])[0]) <= {0, 1}
    assert st["within_tol"] == differ == int(hist[1][1])
    assert st["mismatch"] == st["sign_flip"] == st["nan_inf_asym"] == 0
    assert st["max_ulp"] == 1
    # the float64 sums against torch's float64 reductions (exact terms, wide accumulation)
    d = w.candidate.double() - w.golden.double()
    assert math.isclose(st["sum_abs"], float(d.abs().sum()), rel_tol=1e-12)
    assert math.isclose(st["sum_sq"], float((d * d).sum()), rel_tol=1e-12)


def test_c4_full_size_every_segment(peat_gpu, oracle, h):
    """Full GPT-2-medium list (292 fp16 segments, 354,823,168 pairs) in the
    bench's launch configuration: every segment against the oracle (fanned out
    to the host cores), and the invariants."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c4_gpt2_medium(device="cuda")
    gs, gh = peat_gpu.peat_compare_segmented(h, w.golden, w.candidate, w.offsets, w.rtol, w.atol)
    sizes = np.diff(w.offsets)
    for s in range(len(gs)):
        _check_properties(gs[s], gh[s], int(sizes[s]))
    assert sum(s["nan_inf_asym"] for s in gs) == len(w.meta["nan_inf_positions"])
    gbits, cbits = host_bits(w.golden, "f16"), host_bits(w.candidate, "f16")
    os_, oh = oracle_segmented(gbits, cbits, w.offsets, "f16", w.rtol, w.atol)
    for s in range(len(os_)):
        assert_stats_equal(gs[s], os_[s], f"c4 seg {s}")
    assert_hist_equal(gh, oh, "c4")


def _full_via_segments(peat, oracle, h, w, nseg, ctx):
    """A full-size single tensor in the bench's launch configuration, checked
    through the oracle: the same tensor cut into nseg equal segments is
    compared segment by segment on both sides (bit-exact), and the one-launch
    result must be their exact combination: counts and histograms summed,
    maxima and their lowest indices taken over segments, sums within 1e-10."""
    n = w.n
    off = np.linspace(0, n, nseg + 1).astype(np.int64)
    gb, cb = host_bits(w.golden, w.dtype), host_bits(w.candidate, w.dtype)
    gs, gh = peat.peat_compare_segmented(h, w.golden, w.candidate, off.tolist(), w.rtol, w.atol)
    os_, oh = oracle_segmented(gb, cb, off, w.dtype, w.rtol, w.atol)
    for s in range(nseg):
        assert_stats_equal(gs[s], os_[s], f"{ctx} seg {s}")
    assert_hist_equal(gh, oh, ctx)
    st, hist = peat.peat_compare(h, w.golden, w.candidate, w.rtol, w.atol)
    assert st["n"] == n and st["count"] == [sum(s["count"][k] for s in os_) for k in range(5)]
    assert st["n_finite"] == sum(s["n_finite"] for s in os_)
    assert np.array_equal(hist, oh.sum(axis=0))
    def seg_of(i):
        return int(np.searchsorted(off, i, side="right")) - 1

    def exact(key, i):
        """The exact value (a Fraction) of pair i's quantity behind `key`."""
        if key == "max_ulp":  # an integer: the segment's own maximum is exact
            return os_[seg_of(i)]["max_ulp"]
        gv, cv = value_at(gb, i, w.dtype), value_at(cb, i, w.dtype)
        a = abs(Fraction(cv) - Fraction(gv))
        if key == "max_abs":
            return a
        return a / abs(Fraction(gv)) if gv != 0 else math.inf

    for key, idx in (("max_abs", "argmax_abs"), ("max_rel", "argmax_rel"), ("max_ulp", "argmax_ulp")):
        best = max(s[key] for s in os_ if s[idx] >= 0)
        assert st[key] == best, key
        # the segments whose maximum rounds to the same value; among them the
        # exact maximum (each segment's own argmax holds its exact maximum),
        # and of equal exact values the lowest index, is the only answer
        cands = [int(off[k]) + os_[k][idx] for k in range(nseg) if os_[k][idx] >= 0 and os_[k][key] == best]
        top = max(exact(key, i) for i in cands)
        want = min(i for i in cands if exact(key, i) == top)
        assert st[idx] == want, (key, st[idx], want, cands[:4])
    for key in ("sum_abs", "sum_sq", "sum_signed"):
        total = math.fsum(s[key] for s in os_)
        assert abs(st[key] - total) <= 1e-10 * abs(total) + 1e-300, key
    # the Mean and Variance of Errors scores of the whole tensor, bit for bit,
    # from the segments' exact sums combined exactly
    S1 = sum(s["S1_exact"] for s in os_)
    S2 = sum(s["S2_exact"] for s in os_)
    nf = sum(s["n_finite"] for s in os_)
    assert (st["mean_abs"], st["var_abs"]) == oracle.mean_var(S1, S2, nf)
    return st


def test_c2_full_size_through_the_oracle(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    _full_via_segments(peat_gpu, oracle, h, W.c2_bf16_rne_vs_rtz(device="cuda"), 64, "c2 full")


def test_c5_full_size_through_the_oracle(peat_gpu, oracle, h):
    from paper_2609_13544_gb300 import workloads as W
    w = W.PlaybackSweep(device="cuda").workload(63)
    st = _full_via_segments(peat_gpu, oracle, h, w, 128, "c5 full")
    assert st["n"] == 268_435_456
