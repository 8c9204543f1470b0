"""peat_compare_noalloc (no handle, no allocation) against peat_compare (GPU).

Collected last on purpose: it must pass alone and after every other test,
so it may depend on no state another test leaves (and leaves none: each call
ends with the fixed scratch's accumulator back at zero).
"""
import ctypes

import numpy as np
import pytest

from parity_util import noise_pairs, random_pairs, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0)
    yield handle
    handle.close()


def outputs():
    import torch
    return (torch.full((160,), 0xA5, dtype=torch.uint8, device="cuda"),
            torch.full((128,), -7, dtype=torch.int64, device="cuda"))


def run_both(peat, h, g, c, rtol, atol):
    """The handle path once, then the allocation-free path twice in a row."""
    import torch
    s_ref, h_ref = outputs()
    peat.peat_compare_raw(h, g, c, rtol, atol, s_ref, h_ref)
    got = []
    for _ in range(2):
        s, hh = outputs()
        peat.peat_compare_noalloc_raw(g, c, rtol, atol, s, hh)
        got.append((s, hh))
    torch.cuda.synchronize()
    for s, hh in got:
        assert torch.equal(s, s_ref), "stats differ from peat_compare"
        assert torch.equal(hh, h_ref), "histograms differ from peat_compare"


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("n", [0, 1, 9, 4095, 100003, 3_000_017])
def test_matches_peat_compare_on_two_calls(peat_gpu, h, dtype, n):
    gb, cb = random_pairs(dtype, n, seed=900 + n)
    run_both(peat_gpu, h, to_device(gb, dtype), to_device(cb, dtype), 1e-3, 0.0)


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_matches_on_noise_misaligned_and_with_atol(peat_gpu, h, dtype):
    gb, cb = noise_pairs(dtype, (1 << 21) + 5, seed=31, rel=1e-3)
    run_both(peat_gpu, h, to_device(gb, dtype, 3), to_device(cb, dtype, 3), 2.0 ** -9, 1e-6)


def test_general_list_overflow_matches(peat_gpu, h):
    # random bit patterns: most pairs leave the window, every CTA rescans
    gb, cb = random_pairs("bf16", 12_000_001, seed=77)
    run_both(peat_gpu, h, to_device(gb, "bf16"), to_device(cb, "bf16"), 1e-3, 0.0)


def test_interleaved_with_handle_calls(peat_gpu, h):
    import torch
    gb, cb = noise_pairs("bf16", 1_000_003, seed=5)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    s_ref, h_ref = outputs()
    peat_gpu.peat_compare_raw(h, g, c, 1e-3, 0.0, s_ref, h_ref)
    for _ in range(3):
        s, hh = outputs()
        peat_gpu.peat_compare_noalloc_raw(g, c, 1e-3, 0.0, s, hh)
        s2, h2 = outputs()
        peat_gpu.peat_compare_raw(h, g, c, 1e-3, 0.0, s2, h2)
        torch.cuda.synchronize()
        assert torch.equal(s, s_ref) and torch.equal(hh, h_ref)
        assert torch.equal(s2, s_ref) and torch.equal(h2, h_ref)


def test_rejections_touch_nothing(peat_gpu):
    import torch
    L = peat_gpu.load()
    x = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    s, _ = outputs()
    tol = peat_gpu.Tol(1e-3, 0.0)
    # n beyond the per-SM limit: rejected before any device work
    rc = L.peat_compare_noalloc(x.data_ptr(), x.data_ptr(), 1 << 40, 2, tol, s.data_ptr(), None, None)
    assert rc == 2
    assert "too large" in peat_gpu.peat_last_error(None)
    rc = L.peat_compare_noalloc(x.data_ptr(), x.data_ptr(), 16, 7, tol, s.data_ptr(), None, None)
    assert rc == 1
    rc = L.peat_compare_noalloc(x.data_ptr(), x.data_ptr(), -1, 2, tol, s.data_ptr(), None, None)
    assert rc == 1
    rc = L.peat_compare_noalloc(x.data_ptr(), x.data_ptr(), 16, 2, peat_gpu.Tol(-1.0, 0.0), s.data_ptr(), None,
                                None)
    assert rc == 1
    torch.cuda.synchronize()


def test_expired_wait_marks_the_outputs_and_the_next_call_is_clean(peat_gpu, h):
    """With every bounded wait giving up at once (testing aid), the outputs
    carry the documented mark (argmax fields -2); the status word is cleared
    per call, so the next normal call equals peat_compare again."""
    import torch
    gb, cb = noise_pairs("bf16", 1_000_003, seed=23)
    g, c = to_device(gb, "bf16"), to_device(cb, "bf16")
    peat_gpu.peat_test_noalloc_expire_waits(True)
    try:
        st, _ = peat_gpu.peat_compare_noalloc(g, c, 1e-3, 0.0)
    finally:
        peat_gpu.peat_test_noalloc_expire_waits(False)
    assert st["argmax_abs"] == st["argmax_rel"] == st["argmax_ulp"] == -2
    run_both(peat_gpu, h, g, c, 1e-3, 0.0)
