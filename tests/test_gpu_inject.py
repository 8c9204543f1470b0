"""GPU injector against the oracle's injector: bit-identical outputs and counts."""
import numpy as np
import pytest
import torch

from parity_util import noise_pairs, to_device

pytestmark = pytest.mark.gpu

ITYPE = {"f32": torch.int32, "f16": torch.int16, "bf16": torch.int16}
NPT = {"f32": np.uint32, "f16": np.uint16, "bf16": np.uint16}


@pytest.fixture(scope="module")
def h(peat_gpu):
    handle = peat_gpu.Handle(0)
    yield handle
    handle.close()


def models_for(dtype):
    w = 32 if dtype == "f32" else 16
    ms = [
        [dict(kind="rz", k=5)],
        [dict(kind="rv", k=7)],
        [dict(kind="bitflip", k=16, bit_lo=0, bit_hi=w - 1)],
        [dict(kind="nan_inf", x=1e-3)],
        [dict(kind="signflip", x=1e-2)],
        [dict(kind="rel_gauss", x=1e-3)],
        [dict(kind="add_gauss", x=1e-2)],
        [dict(kind="bias", x=1e-4)],
        [dict(kind="rel_gauss", x=1e-3), dict(kind="signflip", x=1e-3), dict(kind="nan_inf", x=1e-4),
         dict(kind="rv", k=3), dict(kind="rz", k=2)],
    ]
    if dtype == "f32":
        ms += [[dict(kind=k)] for k in ("cast_f16_rne", "cast_f16_rtz", "cast_bf16_rne", "cast_bf16_rtz")]
    return ms


@pytest.mark.parametrize("dtype", ["f32", "f16", "bf16"])
def test_inject_matches_oracle(peat_gpu, oracle, h, dtype):
    n = 200003
    gb, _ = noise_pairs(dtype, n, seed=21, outliers=50)
    src = to_device(gb, dtype)
    for models in models_for(dtype):
        for seed in (0, 12345678901):
            dst, cnt = peat_gpu.peat_pseudo_error_inject(h, src, models, seed)
            got = dst.view(ITYPE[dtype]).cpu().numpy().view(NPT[dtype])
            ref, rcnt = oracle.inject(gb, dtype, [oracle.model(**m) for m in models], seed)
            assert np.array_equal(cnt, rcnt), (models, cnt, rcnt)
            bad = np.nonzero(got != ref)[0]
            assert bad.size == 0, (dtype, models, seed, bad[:5], got[bad[:5]], ref[bad[:5]])


def test_inject_in_place_and_rejections(peat_gpu, oracle, h):
    n = 10007
    gb, _ = noise_pairs("bf16", n, seed=3)
    src = to_device(gb, "bf16")
    models = [dict(kind="rel_gauss", x=1e-2), dict(kind="rv", k=9)]
    out, _ = peat_gpu.peat_pseudo_error_inject(h, src, models, 5, dst=src)
    ref, _ = oracle.inject(gb, "bf16", [oracle.model(**m) for m in models], 5)
    assert np.array_equal(out.view(torch.int16).cpu().numpy().view(np.uint16), ref)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_pseudo_error_inject(h, src, [dict(kind="cast_f16_rne")], 1)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_pseudo_error_inject(h, src, [dict(kind="rz", k=n + 1)], 1)
    with pytest.raises(peat_gpu.PeatError):
        peat_gpu.peat_pseudo_error_inject(h, src, [dict(kind="nan_inf", x=1.5)], 1)
