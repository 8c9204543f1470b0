"""GPU parity on the five synthetic recipes (paper_2609_13544_gb300.workloads).

Oracle-sized cases compare every output; full-size cases, in the launch
configuration the bench times, compare the outputs the oracle can compute one
by one (whole small segments) and check properties that hold at any size.
"""
import math

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


def test_c4_full_size_sampled_segments(peat_gpu, oracle, h):
    """Full GPT-2-medium list: every segment satisfies the invariants; the oracle
    recomputes the 100 smallest segments one by one."""
    from paper_2609_13544_gb300 import workloads as W
    w = W.c4_gpt2_medium(device="cuda")
    gs, gh = peat_gpu.peat_compare_segmented(h, w.golden, w.candidate, w.offsets, w.rtol, w.atol)
    sizes = np.diff(w.offsets)
    for s in range(len(gs)):
        _check_properties(gs[s], gh[s], int(sizes[s]))
    assert sum(s["nan_inf_asym"] for s in gs) == len(w.meta["nan_inf_positions"])
    pick = np.argsort(sizes, kind="stable")[:100]
    gbits, cbits = host_bits(w.golden, "f16"), host_bits(w.candidate, "f16")
    for s in pick:
        a, b = int(w.offsets[s]), int(w.offsets[s + 1])
        os_, oh = oracle.compare(gbits[a:b], cbits[a:b], "f16", w.rtol, w.atol)
        assert_stats_equal(gs[s], os_, f"c4 seg {s}")
        assert_hist_equal(gh[s], oh, f"c4 seg {s}")
