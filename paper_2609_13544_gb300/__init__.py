"""Python binding of libpeat (include/peat.h): argument marshalling only.

Every step of the compare and of the injector runs in the CUDA library;
this module turns torch tensors into device pointers and sizes, calls the C
ABI through ctypes, and unpacks the result records.  It raises if the
library has not been built (there is no CPU fallback).

Names follow the C ABI: ``peat_signature_create``, ``peat_compare``,
``peat_compare_segmented``, ``peat_pseudo_error_inject``, ``peat_inject_compare``, ``peat_last_error``.
"""
from __future__ import annotations

import ctypes
from pathlib import Path
from typing import Optional, Sequence

import numpy as np

from .buildlib import LIB, build  # noqa: F401

DTYPE_CODES = {"f32": 0, "f16": 1, "bf16": 2}
CLASSES = ("exact", "within_tol", "mismatch", "nan_inf_asym", "sign_flip")
HIST_BINS = 128
STATS_BYTES = 160
INJECT_KINDS = {
    "rz": 0, "rv": 1, "bitflip": 2, "nan_inf": 3, "signflip": 4, "rel_gauss": 5,
    "add_gauss": 6, "bias": 7, "cast_f16_rne": 8, "cast_f16_rtz": 9, "cast_bf16_rne": 10,
    "cast_bf16_rtz": 11,
}
PEAT_FLAG_TEST_EXPIRE_WAITS = 0x80000000
STATUS = {0: "PEAT_OK", 1: "PEAT_ERR_INVALID_ARG", 2: "PEAT_ERR_UNSUPPORTED", 3: "PEAT_ERR_ALLOC",
          4: "PEAT_ERR_CUDA", 5: "PEAT_ERR_TIMEOUT", 6: "PEAT_ERR_INTERNAL"}

TOPK_BYTES = 48

# numpy view of peat_topk_t
TOPK_DTYPE = np.dtype([("n_finite", "<u8"), ("k", "<u8"), ("threshold", "<f8"), ("sum", "<f8"), ("mean", "<f8"),
                       ("exact", "<u4"), ("reserved", "<u4")])
assert TOPK_DTYPE.itemsize == TOPK_BYTES

TSTATS_BYTES = 80

# numpy view of peat_tstats_t
TSTATS_DTYPE = np.dtype([("n", "<u8"), ("n_finite", "<u8"), ("n_nan", "<u8"), ("n_inf", "<u8"), ("sum", "<f8"),
                         ("sum_sq", "<f8"), ("mean", "<f8"), ("var", "<f8"), ("min", "<f8"), ("max", "<f8")])
assert TSTATS_DTYPE.itemsize == TSTATS_BYTES

# numpy view of peat_stats_t
STATS_DTYPE = np.dtype([
    ("n", "<u8"), ("count", "<u8", (5,)), ("n_finite", "<u8"),
    ("max_abs", "<f8"), ("argmax_abs", "<i8"), ("max_rel", "<f8"), ("argmax_rel", "<i8"),
    ("max_ulp", "<u8"), ("argmax_ulp", "<i8"), ("sum_abs", "<f8"), ("sum_sq", "<f8"),
    ("sum_signed", "<f8"), ("rtol_eff", "<f8"), ("atol_eff", "<f8"), ("mean_abs", "<f8"), ("var_abs", "<f8"),
])
assert STATS_DTYPE.itemsize == STATS_BYTES


class PeatError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [("device", ctypes.c_int32), ("reserved0", ctypes.c_int32), ("max_segments", ctypes.c_int64),
                ("flags", ctypes.c_uint32), ("reserved1", ctypes.c_uint32)]


class Tol(ctypes.Structure):
    _fields_ = [("rtol", ctypes.c_double), ("atol", ctypes.c_double)]


class InjectModel(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("k", ctypes.c_int32), ("bit_lo", ctypes.c_int32),
                ("bit_hi", ctypes.c_int32), ("x", ctypes.c_double)]


EXPORTS = ("peat_signature_create", "peat_signature_destroy", "peat_compare", "peat_compare_segmented",
           "peat_pseudo_error_inject", "peat_last_error", "peat_compare_noalloc", "peat_topk_mean",
           "peat_tensor_stats", "peat_spearman", "peat_mean_std", "peat_isclose_grid", "peat_inject_compare",
           "peat_test_noalloc_expire_waits", "peat_test_for_digits", "peat_trend", "peat_set_stage1_event",
           "peat_test_quot_rn")

_lib: Optional[ctypes.CDLL] = None


def load(path: Optional[Path] = None) -> ctypes.CDLL:
    """Load libpeat.so; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    p = Path(path) if path else LIB
    if not p.exists():
        raise RuntimeError(f"{p} is missing: build it with paper_2609_13544_gb300.buildlib.build() "
                           "(or __graft_entry__.build()); there is no fallback")
    L = ctypes.CDLL(str(p))
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    L.peat_signature_create.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(Config)]
    L.peat_signature_create.restype = i32
    L.peat_signature_destroy.argtypes = [vp]
    L.peat_signature_destroy.restype = i32
    L.peat_compare.argtypes = [vp, vp, vp, i64, i32, Tol, vp, vp, vp]
    L.peat_compare.restype = i32
    L.peat_compare_segmented.argtypes = [vp, vp, vp, vp, i64, i32, Tol, vp, vp, vp]
    L.peat_compare_segmented.restype = i32
    L.peat_pseudo_error_inject.argtypes = [vp, vp, vp, i64, i32, ctypes.POINTER(InjectModel), i32,
                                           ctypes.c_uint64, vp, vp]
    L.peat_pseudo_error_inject.restype = i32
    L.peat_inject_compare.argtypes = [vp, vp, i64, i32, ctypes.POINTER(InjectModel), i32, ctypes.c_uint64, Tol,
                                      vp, vp, vp]
    L.peat_inject_compare.restype = i32
    L.peat_last_error.argtypes = [vp]
    L.peat_last_error.restype = ctypes.c_char_p
    L.peat_compare_noalloc.argtypes = [vp, vp, i64, i32, Tol, vp, vp, vp]
    L.peat_compare_noalloc.restype = i32
    L.peat_test_noalloc_expire_waits.argtypes = [i32]
    L.peat_test_noalloc_expire_waits.restype = None
    L.peat_test_for_digits.argtypes = [ctypes.c_uint64, ctypes.c_uint64, i32, i32, ctypes.c_void_p]
    L.peat_test_for_digits.restype = i32
    L.peat_trend.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p,
                             ctypes.c_void_p, ctypes.c_void_p]
    L.peat_trend.restype = i32
    L.peat_set_stage1_event.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    L.peat_set_stage1_event.restype = i32
    L.peat_test_quot_rn.argtypes = [ctypes.c_uint64, ctypes.c_uint64, i32, i32, ctypes.c_uint64]
    L.peat_test_quot_rn.restype = ctypes.c_double
    L.peat_topk_mean.argtypes = [vp, vp, vp, i64, i32, ctypes.c_uint64, ctypes.c_uint64, vp, vp]
    L.peat_topk_mean.restype = i32
    L.peat_isclose_grid.argtypes = [vp, vp, vp, i64, i32, vp, i32, vp, i32, vp, vp]
    L.peat_isclose_grid.restype = i32
    L.peat_tensor_stats.argtypes = [vp, vp, vp, i64, i32, vp, vp]
    L.peat_tensor_stats.restype = i32
    dp = ctypes.POINTER(ctypes.c_double)
    L.peat_spearman.argtypes = [dp, dp, i64, dp]
    L.peat_spearman.restype = i32
    L.peat_mean_std.argtypes = [dp, i64, i32, dp, dp]
    L.peat_mean_std.restype = i32
    _lib = L
    return L


def peat_last_error(h=None) -> str:
    return load().peat_last_error(h.ptr if isinstance(h, Handle) else h).decode()


def _check(rc: int, h) -> None:
    if rc != 0:
        raise PeatError(rc, peat_last_error(h))


class Handle:
    """Owns one peat_handle_t (peat_signature_create / peat_signature_destroy)."""

    def __init__(self, device: int = 0, max_segments: int = 0, flags: int = 0):
        self.ptr = ctypes.c_void_p()
        cfg = Config(device, 0, max_segments, flags, 0)
        _check(load().peat_signature_create(ctypes.byref(self.ptr), ctypes.byref(cfg)), None)
        self.device = device

    def close(self) -> None:
        if self.ptr:
            load().peat_signature_destroy(self.ptr)
            self.ptr = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()


def peat_signature_create(device: int = 0, max_segments: int = 0, flags: int = 0) -> Handle:
    return Handle(device, max_segments, flags)


def peat_signature_destroy(h: Handle) -> None:
    h.close()


def dtype_code(t) -> int:
    import torch
    m = {torch.float32: 0, torch.float16: 1, torch.bfloat16: 2, torch.float8_e4m3fn: 3, torch.float8_e5m2: 4,
         torch.float64: 5}
    if t.dtype not in m:
        raise TypeError(f"unsupported dtype {t.dtype}")
    return m[t.dtype]


def _stream_ptr(stream) -> Optional[int]:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _sync(stream) -> None:
    """The dict wrappers read their outputs back: wait for the stream the call ran on."""
    if stream is not None:
        stream.synchronize()


def _dev_tensor_check(*ts):
    for t in ts:
        if not t.is_cuda:
            raise ValueError("golden/candidate must be CUDA tensors")
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")


def peat_compare_raw(h: Handle, golden, candidate, rtol: float, atol: float, stats_out, hist_out=None,
                     stream=None) -> None:
    """peat_compare on preallocated device outputs (stats_out: uint8[160], hist_out: int64[128])."""
    _dev_tensor_check(golden, candidate)
    if golden.numel() != candidate.numel() or golden.dtype != candidate.dtype:
        raise ValueError("golden and candidate differ in size or dtype")
    rc = load().peat_compare(h.ptr, golden.data_ptr(), candidate.data_ptr(), golden.numel(), dtype_code(golden),
                             Tol(rtol, atol), stats_out.data_ptr(),
                             hist_out.data_ptr() if hist_out is not None else None, _stream_ptr(stream))
    _check(rc, h)


def peat_compare_noalloc_raw(golden, candidate, rtol: float, atol: float, stats_out, hist_out=None,
                             stream=None) -> None:
    """peat_compare_noalloc (no handle, no allocation) on preallocated device outputs."""
    _dev_tensor_check(golden, candidate)
    if golden.numel() != candidate.numel() or golden.dtype != candidate.dtype:
        raise ValueError("golden and candidate differ in size or dtype")
    rc = load().peat_compare_noalloc(golden.data_ptr(), candidate.data_ptr(), golden.numel(), dtype_code(golden),
                                     Tol(rtol, atol), stats_out.data_ptr(),
                                     hist_out.data_ptr() if hist_out is not None else None, _stream_ptr(stream))
    _check(rc, None)


def peat_compare_segmented_raw(h: Handle, golden, candidate, offsets, rtol: float, atol: float, stats_out,
                               hist_out=None, stream=None) -> None:
    _dev_tensor_check(golden, candidate)
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    if golden.numel() != candidate.numel() or golden.dtype != candidate.dtype:
        raise ValueError("golden and candidate differ in size or dtype")
    if off.size < 1 or off[-1] > golden.numel():
        raise ValueError("offsets exceed the tensors")
    rc = load().peat_compare_segmented(h.ptr, golden.data_ptr(), candidate.data_ptr(), off.ctypes.data,
                                       off.size - 1, dtype_code(golden), Tol(rtol, atol), stats_out.data_ptr(),
                                       hist_out.data_ptr() if hist_out is not None else None,
                                       _stream_ptr(stream))
    _check(rc, h)


def stats_to_dicts(raw: np.ndarray) -> list:
    """Unpack host bytes (k*160) into dicts, one per peat_stats_t record."""
    arr = np.frombuffer(np.ascontiguousarray(raw).tobytes(), dtype=STATS_DTYPE)
    out = []
    for r in arr:
        d = {k: (r[k].item() if k != "count" else [int(v) for v in r[k]]) for k in STATS_DTYPE.names}
        for name, v in zip(CLASSES, d["count"]):
            d[name] = v
        out.append(d)
    return out


def peat_compare(h: Handle, golden, candidate, rtol: float, atol: float = 0.0, stream=None):
    """Signature of one tensor pair: (stats dict, hist numpy uint64[2, 64]); synchronises."""
    import torch
    dev = golden.device
    stats = torch.empty(STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(HIST_BINS, dtype=torch.int64, device=dev)
    peat_compare_raw(h, golden, candidate, rtol, atol, stats, hist, stream)
    _sync(stream)
    s = stats_to_dicts(stats.cpu().numpy())[0]
    return s, hist.cpu().numpy().view(np.uint64).reshape(2, 64)


def peat_test_noalloc_expire_waits(on: bool) -> None:
    """Testing aid: every bounded device-side wait of later peat_compare_noalloc calls gives up at once."""
    load().peat_test_noalloc_expire_waits(1 if on else 0)


def peat_test_for_digits(m: int, e: int, neg: bool):
    """Testing aid (host only): the kernels' digit split of +-m 2^e -> (24 signed
    digits of weight 2^(32 j - 416), True if a digit fell outside them)."""
    out = np.zeros(24, np.int64)
    rc = load().peat_test_for_digits(m & (2 ** 64 - 1), m >> 64, int(e), 1 if neg else 0, out.ctypes.data)
    return out, rc == 1


def peat_compare_noalloc(golden, candidate, rtol: float, atol: float = 0.0, stream=None):
    """peat_compare_noalloc of one tensor pair: (stats dict, hist numpy uint64[2, 64]); synchronises.
    (This convenience wrapper allocates its output tensors; the C entry point itself allocates nothing.)"""
    import torch
    dev = golden.device
    stats = torch.empty(STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(HIST_BINS, dtype=torch.int64, device=dev)
    peat_compare_noalloc_raw(golden, candidate, rtol, atol, stats, hist, stream)
    _sync(stream)
    s = stats_to_dicts(stats.cpu().numpy())[0]
    return s, hist.cpu().numpy().view(np.uint64).reshape(2, 64)


def peat_compare_segmented(h: Handle, golden, candidate, offsets: Sequence[int], rtol: float, atol: float = 0.0,
                           stream=None):
    """Per-segment signatures: (list of dicts, hist numpy uint64[nseg, 2, 64]); synchronises."""
    import torch
    dev = golden.device
    nseg = len(offsets) - 1
    stats = torch.empty(max(nseg, 1) * STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(max(nseg, 1) * HIST_BINS, dtype=torch.int64, device=dev)
    peat_compare_segmented_raw(h, golden, candidate, offsets, rtol, atol, stats, hist, stream)
    _sync(stream)
    if nseg == 0:
        return [], np.zeros((0, 2, 64), np.uint64)
    s = stats_to_dicts(stats.cpu().numpy()[: nseg * STATS_BYTES])
    return s, hist.cpu().numpy()[: nseg * HIST_BINS].view(np.uint64).reshape(nseg, 2, 64)


def peat_topk_mean_raw(h: Handle, golden, candidate, num: int, den: int, out, stream=None) -> None:
    """peat_topk_mean on a preallocated device output (out: uint8[48])."""
    _dev_tensor_check(golden, candidate)
    if golden.numel() != candidate.numel() or golden.dtype != candidate.dtype:
        raise ValueError("golden and candidate differ in size or dtype")
    rc = load().peat_topk_mean(h.ptr, golden.data_ptr(), candidate.data_ptr(), golden.numel(), dtype_code(golden),
                               ctypes.c_uint64(num), ctypes.c_uint64(den), out.data_ptr(), _stream_ptr(stream))
    _check(rc, h)


def peat_topk_mean(h: Handle, golden, candidate, num: int = 1, den: int = 10, stream=None) -> dict:
    """Mean of the top num/den of the errors of one tensor pair: dict of n_finite, k,
    threshold, sum, mean, exact; synchronises."""
    import torch
    out = torch.empty(TOPK_BYTES, dtype=torch.uint8, device=golden.device)
    peat_topk_mean_raw(h, golden, candidate, num, den, out, stream)
    _sync(stream)
    r = np.frombuffer(out.cpu().numpy().tobytes(), dtype=TOPK_DTYPE)[0]
    return {k: r[k].item() for k in TOPK_DTYPE.names if k != "reserved"}


def peat_tensor_stats_raw(h: Handle, x, offsets, stats_out, stream=None) -> None:
    """peat_tensor_stats on a preallocated device output (stats_out: uint8[80 * nseg])."""
    _dev_tensor_check(x)
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    if off.size < 1 or off[-1] > x.numel():
        raise ValueError("offsets exceed the tensor")
    rc = load().peat_tensor_stats(h.ptr, x.data_ptr(), off.ctypes.data, off.size - 1, dtype_code(x),
                                  stats_out.data_ptr(), _stream_ptr(stream))
    _check(rc, h)


def peat_tensor_stats(h: Handle, x, offsets: Optional[Sequence[int]] = None, stream=None):
    """Context statistics of x (one dict) or of each segment (a list of dicts); synchronises."""
    import torch
    off = [0, x.numel()] if offsets is None else list(offsets)
    nseg = len(off) - 1
    out = torch.empty(max(nseg, 1) * TSTATS_BYTES, dtype=torch.uint8, device=x.device)
    peat_tensor_stats_raw(h, x, off, out, stream)
    _sync(stream)
    arr = np.frombuffer(out.cpu().numpy()[: nseg * TSTATS_BYTES].tobytes(), dtype=TSTATS_DTYPE)
    res = [{k: r[k].item() for k in TSTATS_DTYPE.names} for r in arr]
    return res[0] if offsets is None else res


def peat_isclose_grid_raw(h: Handle, golden, candidate, rtols, atols, counts_out, stream=None) -> None:
    """peat_isclose_grid on a preallocated device output (counts_out: int64[len(rtols) * len(atols)])."""
    _dev_tensor_check(golden, candidate)
    if golden.numel() != candidate.numel() or golden.dtype != candidate.dtype:
        raise ValueError("golden and candidate differ in size or dtype")
    r, a = _host_doubles(rtols), _host_doubles(atols)
    rc = load().peat_isclose_grid(h.ptr, golden.data_ptr(), candidate.data_ptr(), golden.numel(),
                                  dtype_code(golden), r.ctypes.data, r.size, a.ctypes.data, a.size,
                                  counts_out.data_ptr(), _stream_ptr(stream))
    _check(rc, h)


def peat_isclose_grid(h: Handle, golden, candidate, rtols, atols, stream=None) -> np.ndarray:
    """isclose pass counts, uint64 [len(rtols), len(atols)]; synchronises."""
    import torch
    out = torch.empty(len(rtols) * len(atols), dtype=torch.int64, device=golden.device)
    peat_isclose_grid_raw(h, golden, candidate, rtols, atols, out, stream)
    _sync(stream)
    return out.cpu().numpy().view(np.uint64).reshape(len(rtols), len(atols))


def _host_doubles(v) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(v, dtype=np.float64))


def peat_spearman(x, y) -> float:
    """Spearman rank correlation of two host sequences (mean ranks for ties)."""
    a, b = _host_doubles(x), _host_doubles(y)
    if a.size != b.size:
        raise ValueError("x and y differ in length")
    dp = ctypes.POINTER(ctypes.c_double)
    rho = ctypes.c_double()
    rc = load().peat_spearman(a.ctypes.data_as(dp), b.ctypes.data_as(dp), a.size, ctypes.byref(rho))
    _check(rc, None)
    return rho.value


def peat_mean_std(x, ddof: int = 0):
    """(mean, std) of a host sequence of scores (ddof 0: population, 1: sample)."""
    a = _host_doubles(x)
    dp = ctypes.POINTER(ctypes.c_double)
    m, sd = ctypes.c_double(), ctypes.c_double()
    rc = load().peat_mean_std(a.ctypes.data_as(dp), a.size, ddof, ctypes.byref(m), ctypes.byref(sd))
    _check(rc, None)
    return m.value, sd.value


def peat_set_stage1_event(h: Handle, event) -> None:
    """Profiling aid: record `event` (a torch.cuda.Event that has been recorded
    once, so that it exists; None: stop) after each later compare's stage-1 launch."""
    ptr = None if event is None else ctypes.c_void_p(event.cuda_event)
    _check(load().peat_set_stage1_event(h.ptr, ptr), h)


def peat_test_quot_rn(W: int, sticky: bool, e: int, d: int) -> float:
    """Testing aid (host only): the kernels' RN-even binary64 of (W + f) 2^e / d."""
    return load().peat_test_quot_rn(W >> 64, W & (2 ** 64 - 1), 1 if sticky else 0, int(e), int(d))


def peat_trend(x, y) -> dict:
    """Least-squares power-law trend of y against x (log y = intercept + slope log x)
    over the points with both values finite and positive: dict of slope,
    intercept, r2 and used (the number of points kept)."""
    a, b = _host_doubles(x), _host_doubles(y)
    if a.size != b.size:
        raise ValueError("x and y differ in length")
    sl, ic, r2 = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
    used = ctypes.c_int64()
    rc = load().peat_trend(a.ctypes.data, b.ctypes.data, a.size, ctypes.byref(sl), ctypes.byref(ic),
                           ctypes.byref(r2), ctypes.byref(used))
    _check(rc, None)
    return {"slope": sl.value, "intercept": ic.value, "r2": r2.value, "used": used.value}


def inject_model(kind: str, k: int = 0, bit_lo: int = 0, bit_hi: int = 0, x: float = 0.0) -> dict:
    return {"kind": kind, "k": k, "bit_lo": bit_lo, "bit_hi": bit_hi, "x": x}


def peat_pseudo_error_inject_raw(h: Handle, dst, src, models: Sequence[dict], seed: int, counts_out,
                                 stream=None) -> None:
    """peat_pseudo_error_inject on preallocated device tensors (counts_out: int64[len(models)])."""
    _dev_tensor_check(dst, src)
    if dst.numel() != src.numel() or dst.dtype != src.dtype:
        raise ValueError("dst and src differ in size or dtype")
    rc = load().peat_pseudo_error_inject(h.ptr, dst.data_ptr(), src.data_ptr(), src.numel(), dtype_code(src),
                                         _model_array(models), len(models), ctypes.c_uint64(seed),
                                         counts_out.data_ptr(), _stream_ptr(stream))
    _check(rc, h)


def peat_pseudo_error_inject(h: Handle, src, models: Sequence[dict], seed: int, dst=None, stream=None):
    """Apply error models to src on the GPU; returns (dst tensor, counts numpy uint64)."""
    import torch
    _dev_tensor_check(src)
    if dst is None:
        dst = torch.empty_like(src)
    arr = _model_array(models)
    counts = torch.zeros(max(len(models), 1), dtype=torch.int64, device=src.device)
    rc = load().peat_pseudo_error_inject(h.ptr, dst.data_ptr(), src.data_ptr(), src.numel(), dtype_code(src), arr,
                                         len(models), ctypes.c_uint64(seed), counts.data_ptr(),
                                         _stream_ptr(stream))
    _check(rc, h)
    _sync(stream)
    return dst, counts[: len(models)].cpu().numpy().view(np.uint64)


def _model_array(models: Sequence[dict]):
    arr = (InjectModel * max(len(models), 1))()
    for i, m in enumerate(models):
        arr[i] = InjectModel(INJECT_KINDS[m["kind"]], m.get("k", 0), m.get("bit_lo", 0), m.get("bit_hi", 0),
                             float(m.get("x", 0.0)))
    return arr


def peat_inject_compare_raw(h: Handle, golden, models: Sequence[dict], seed: int, rtol: float, atol: float,
                            stats_out, hist_out=None, stream=None) -> None:
    """peat_inject_compare on preallocated device outputs (stats_out: uint8[160], hist_out: int64[128])."""
    _dev_tensor_check(golden)
    rc = load().peat_inject_compare(h.ptr, golden.data_ptr(), golden.numel(), dtype_code(golden),
                                    _model_array(models), len(models), ctypes.c_uint64(seed), Tol(rtol, atol),
                                    stats_out.data_ptr(), hist_out.data_ptr() if hist_out is not None else None,
                                    _stream_ptr(stream))
    _check(rc, h)


def peat_inject_compare(h: Handle, golden, models: Sequence[dict], seed: int, rtol: float, atol: float = 0.0,
                        stream=None):
    """Signature of golden against its injected copy (generated in the kernel, never stored):
    (stats dict, hist numpy uint64[2, 64]); synchronises."""
    import torch
    dev = golden.device
    stats = torch.empty(STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(HIST_BINS, dtype=torch.int64, device=dev)
    peat_inject_compare_raw(h, golden, models, seed, rtol, atol, stats, hist, stream)
    _sync(stream)
    s = stats_to_dicts(stats.cpu().numpy())[0]
    return s, hist.cpu().numpy().view(np.uint64).reshape(2, 64)


def derived_scores(st: dict) -> dict:
    """The scores of Section IV-B-3 from one signature.  Max, Mean and Variance
    of |e| are the record's own fields (the mean and the variance computed on
    the device, exact and rounded once); bias, L2 and RMS are conveniences
    derived here from the rounded sums."""
    import math
    nf = st["n_finite"]
    return {"max": st["max_abs"], "mean": st["mean_abs"], "var": st["var_abs"],
            "bias": st["sum_signed"] / nf if nf else 0.0, "l2": math.sqrt(st["sum_sq"]),
            "rms": math.sqrt(st["sum_sq"] / nf) if nf else 0.0}
