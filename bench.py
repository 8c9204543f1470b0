"""Throughput of the golden-vs-candidate error signature (peat_compare) on GB300.

One step = one full call of the compare over one synthetic workload resident
in HBM: both tensors streamed once, every segment's signature finalized (in
the same kernel for a single-segment call, by a second small launch for a
segmented one).
Default workload: the [8,2048,4096] bf16 activation (67,108,864 pairs,
RNE vs RTZ candidate).  Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c1..c5] [--impl reference]

For N > 1 it runs under torch.distributed.run, one rank per GPU; every rank
compares its own copy of the workload (weak scaling: the compare of one
tensor is independent per rank, no data-path collective); time = max over
ranks between barriers.
"""
from __future__ import annotations

import argparse
import gc
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "element-pairs/s and achieved HBM GB/s (fraction of ~8 TB/s) for peat_compare"
WORKLOAD_NAMES = {
    "c1": "single fp32 tensor n=1,048,576, N(0,1) golden, rel noise 1e-6 + 16 bit flips, rtol 1e-5",
    "c2": "bf16 activation [8,2048,4096] (67,108,864 pairs): RNE vs RTZ rounding of N(0,2^2) fp32, rtol 2^-7",
    "c3": "ResNet-50 parameter list, 161 fp32 segments (25,557,032 pairs), Kaiming-normal, bias/noise candidate",
    "c4": "GPT-2-medium parameter list, 292 fp16 segments (354,823,168 pairs), Laplace(0,0.02), noise+NaN/Inf+sign flips",
    "c5": "playback sweep step 63 of a 268,435,456-element bf16 tensor, rel noise 1e-4*sqrt(s)",
}
NOMINAL_HBM_GBS = 8000.0


def measured_peaks() -> dict:
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        return json.loads(p.read_text())
    return {"hbm_gbs": 6800.0, "fallback": True}


def kernel_source_sha() -> str:
    h = hashlib.sha256()
    for f in ("compare.cu", "exact.cuh", "meanvar.cuh", "inject_models.cuh", "peat_internal.h"):
        h.update((ROOT / "paper_2609_13544_gb300" / "csrc" / f).read_bytes())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str):
    """DRAM bytes per stage-1 launch from the committed ncu summary, if it was
    taken on the current kernel source."""
    p = ROOT / "profiles" / "traffic.json"
    if not p.exists():
        return None
    d = json.loads(p.read_text()).get(workload)
    if not d or d.get("source_sha") != kernel_source_sha():
        return None
    return d.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 200 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = Path(os.environ.get("TMPDIR", "/tmp")) / f"peat_clocks_{os.getpid()}.csv"

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self) -> dict:
        if self.proc is None or not self.path.exists():
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in self.path.read_text().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(parts)
            except ValueError:
                pass
        self.path.unlink(missing_ok=True)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


class NvmlSampler:
    """SM clock, its maximum, power and the clock event reasons of one GPU,
    read in-process through NVML (read-only queries) every `period` seconds
    on a background thread.  The GPU is found by the PCI bus id the CUDA
    driver reports for the process's device (CUDA and NVML ordinals differ
    under CUDA_VISIBLE_DEVICES).  available is False when NVML or the CUDA
    driver library cannot be loaded; the caller then falls back to
    nvidia-smi."""
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
               0x80: "hw_power_brake_slowdown", 0x2: "applications_clocks_setting"}

    def __init__(self, cuda_ordinal: int, period: float = 0.01):
        import ctypes
        import threading
        self.period = period
        self.rows = []
        self.available = False
        self._stop = threading.Event()
        self._thread = None
        try:
            self.nv = ctypes.CDLL("libnvidia-ml.so.1")
            cu = ctypes.CDLL("libcuda.so.1")
            if cu.cuInit(0) != 0:
                return
            dev = ctypes.c_int()
            if cu.cuDeviceGet(ctypes.byref(dev), cuda_ordinal) != 0:
                return
            bus = ctypes.create_string_buffer(64)
            if cu.cuDeviceGetPCIBusId(bus, 64, dev) != 0:
                return
            if self.nv.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if self.nv.nvmlDeviceGetHandleByPciBusId_v2(bus, ctypes.byref(self.h)) != 0:
                return
            mx = ctypes.c_uint()
            self.max_mhz = mx.value if self.nv.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx)) == 0 else None
            self.reasons_fn = getattr(self.nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(self.nv, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.available = True
        except (OSError, AttributeError):
            self.available = False

    def sample(self):
        import ctypes
        mhz, mw, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        ok = self.nv.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(mhz)) == 0  # NVML_CLOCK_SM
        self.nv.nvmlDeviceGetPowerUsage(self.h, ctypes.byref(mw))
        self.reasons_fn(self.h, ctypes.byref(rs))
        if ok:
            self.rows.append((time.perf_counter(), mhz.value, mw.value / 1000.0, rs.value))

    def _run(self):
        while not self._stop.is_set():
            self.sample()
            self._stop.wait(self.period)

    def __enter__(self):
        import threading
        self.rows = []
        if self.available:
            self._stop.clear()
            self._thread = threading.Thread(target=self._run, daemon=True)
            self._thread.start()
        return self

    def __exit__(self, *a):
        if self._thread is not None:
            self._stop.set()
            self._thread.join()
            self.sample()

    def summary(self, t0=None, t1=None) -> dict:
        rows = [r for r in self.rows if (t0 is None or r[0] >= t0) and (t1 is None or r[0] <= t1)] or self.rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0, "source": "nvml"}
        busy = [r for r in rows if not (r[3] & 0x1)] or rows  # samples not flagged idle
        reasons = sorted({name for r in busy for bit, name in self.REASONS.items() if r[3] & bit})
        return {"sm_mhz": statistics.median(r[1] for r in busy), "sm_max_mhz": self.max_mhz,
                "sm_mhz_min": min(r[1] for r in busy), "power_w_max": max(r[2] for r in rows),
                "reasons": reasons, "samples": len(rows), "samples_not_idle": len(busy),
                "period_ms": self.period * 1e3, "source": "nvml in-process (read-only queries)"}


def make_workload(name: str, device: str):
    from paper_2609_13544_gb300 import workloads as W
    if name == "c1":
        return W.c1_single_fp32(device=device)
    if name == "c2":
        return W.c2_bf16_rne_vs_rtz(device=device)
    if name == "c3":
        return W.c3_resnet50(device=device)
    if name == "c4":
        return W.c4_gpt2_medium(device=device)
    if name == "c5":
        return W.PlaybackSweep(device=device).workload(63)
    raise ValueError(name)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(x: float, device) -> float:
    """The slowest replica sets the step time: MAX over ranks (identity at N = 1)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, steps: int, ms: float) -> float:
    """Units all ranks processed in `steps` steps, per second of the max-over-ranks time."""
    return units_per_rank * world * steps / (ms * 1e-3)


# --------------------------------------------------------------------------- oracle timing
def _oracle_slice(args):
    import numpy as np
    import oracle
    g, c, dtype, rtol, atol, segs = args
    t0 = time.perf_counter()
    if segs is None:
        oracle.compare(g, c, dtype, rtol, atol)
    else:
        oracle.compare_segmented(g, c, segs, dtype, rtol, atol)
    return time.perf_counter() - t0


def host_bits(t, dtype):
    import numpy as np
    import torch
    it = torch.int32 if dtype == "f32" else torch.int16
    return t.contiguous().view(it).cpu().numpy().view(np.uint32 if dtype == "f32" else np.uint16)


def oracle_rate(w, pool, cores: int, pairs: int) -> tuple:
    """Oracle pairs/s on the first `pairs` pairs, split across `cores` processes."""
    import numpy as np
    pairs = min(pairs, w.n)
    gb, cb = host_bits(w.golden[:pairs], w.dtype), host_bits(w.candidate[:pairs], w.dtype)
    bounds = np.linspace(0, pairs, cores + 1).astype(np.int64)
    jobs = [(gb[a:b], cb[a:b], w.dtype, w.rtol, w.atol, None) for a, b in zip(bounds[:-1], bounds[1:]) if b > a]
    t0 = time.perf_counter()
    list(pool.map(_oracle_slice, jobs))
    dt = time.perf_counter() - t0
    return pairs / dt, dt, pairs


def make_pool(cores):
    import multiprocessing as mp
    from concurrent.futures import ProcessPoolExecutor
    return ProcessPoolExecutor(max_workers=cores, mp_context=mp.get_context("spawn"))


def run_reference(args) -> None:
    """Reference arm: the oracle, as it stands, on the host cores."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import oracle
    oracle.build()
    w = make_workload(args.workload, "cpu")
    cores = os.cpu_count() or 1
    with make_pool(cores) as pool:
        # size each step's sample so the whole run stays within about a minute of wall time
        rate, _, _ = oracle_rate(w, pool, cores, min(w.n, 200_000 * cores))
        per_step = int(max(4096 * cores, min(w.n, rate * 60.0 / max(1, args.steps + args.warmup))))
        for _ in range(args.warmup):
            oracle_rate(w, pool, cores, per_step)
        t0 = time.perf_counter()
        done = 0
        for _ in range(args.steps):
            _, _, p = oracle_rate(w, pool, cores, per_step)
            done += p
        dt = time.perf_counter() - t0
    value = done / dt
    sample = f"first {per_step} pairs of {args.workload} per step, split over {cores} processes"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "pairs/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / max(1, args.steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64+exact int",
        "data": "synthetic",
        "config": {"workload": WORKLOAD_NAMES[args.workload], "element": w.dtype, "pairs_per_step": per_step},
        "cpu_baseline": {"value": value, "unit": "pairs/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "pairs/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- oracle sample + parity
INT_KEYS = ("n", "count", "n_finite", "argmax_abs", "argmax_rel", "max_ulp", "argmax_ulp")
EXACT_KEYS = ("max_abs", "max_rel", "rtol_eff", "atol_eff", "mean_abs", "var_abs")
SUM_KEYS = ("sum_abs", "sum_sq", "sum_signed")


def _oracle_job(args):
    import oracle
    g, c, offs, dtype, rtol, atol = args
    t0 = time.perf_counter()
    st, hist = oracle.compare_segmented(g, c, offs, dtype, rtol, atol)
    for d in st:  # the exact sums are Fractions; only the rounded outputs travel back
        d.pop("S1_exact", None)
        d.pop("S2_exact", None)
    return time.perf_counter() - t0, st, hist


def oracle_sample(w, pool, cores: int, pairs: int):
    """The oracle on the first `pairs` pairs of a workload, cut at the
    workload's own segment boundaries and at `cores` equal chunks (one
    process each): (pairs/s, seconds, pairs, cut offsets, stats, hist)."""
    import numpy as np
    P = int(min(pairs, w.n))
    chunks = np.linspace(0, P, cores + 1).astype(np.int64)
    cuts = set(int(x) for x in chunks)
    if w.offsets is not None:
        cuts |= {int(o) for o in w.offsets if 0 <= int(o) <= P}
    off = np.array(sorted(cuts), np.int64)
    gb, cb = host_bits(w.golden[:P], w.dtype), host_bits(w.candidate[:P], w.dtype)
    jobs = []
    for a, b in zip(chunks[:-1], chunks[1:]):
        if b > a:
            sub = off[(off >= a) & (off <= b)]
            jobs.append((gb[a:b], cb[a:b], sub - a, w.dtype, w.rtol, w.atol))
    t0 = time.perf_counter()
    res = list(pool.map(_oracle_job, jobs))
    dt = time.perf_counter() - t0
    stats = [d for r in res for d in r[1]]
    hist = np.concatenate([r[2] for r in res])
    return P / dt, dt, P, off, stats, hist


def parity_on_sample(peat, h, w, off, ostats, ohist) -> dict:
    """The CUDA path on the oracle's sample, cut the same way (one segmented
    call): every integer output and maximum bit for bit, the binary64 sums
    within 1e-10 relative."""
    import numpy as np
    P = int(off[-1])
    gs, gh = peat.peat_compare_segmented(h, w.golden[:P], w.candidate[:P], off.tolist(), w.rtol, w.atol)
    bad = None
    for k, (a, b) in enumerate(zip(gs, ostats)):
        for key in INT_KEYS + EXACT_KEYS:
            if a[key] != b[key]:
                bad = bad or f"segment {k}: {key} gpu={a[key]!r} oracle={b[key]!r}"
        for key in SUM_KEYS:
            if not (a[key] == b[key] or abs(a[key] - b[key]) <= 1e-10 * abs(b[key])):
                bad = bad or f"segment {k}: {key} gpu={a[key]!r} oracle={b[key]!r}"
    if not np.array_equal(np.asarray(gh), np.asarray(ohist)):
        bad = bad or "histograms differ"
    return {"status": "ok" if bad is None else "MISMATCH", "pairs": P, "segments": len(gs),
            "checked": "counts, maxima, argmax, mean/var bit for bit; sums within 1e-10; both histograms",
            **({"first_mismatch": bad} if bad else {})}


# --------------------------------------------------------------------------- per-config timings
def events_ms(torch, stream, fn, calls: int) -> float:
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(calls):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / calls


def config_block(peat, h, name: str, w, stream, peak: float, cold: bool) -> dict:
    """Hot timing (back-to-back calls, about 50 ms of them), cold timing with
    L2 flushed between calls (a 512 MiB write) where asked, and for a
    segmented call stage 1 alone against stage 1 + the finalize."""
    import torch
    nseg = 1 if w.offsets is None else len(w.offsets) - 1
    dev = w.golden.device
    stats = torch.empty(nseg * peat.STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(nseg * peat.HIST_BINS, dtype=torch.int64, device=dev)

    def call():
        if w.offsets is None:
            peat.peat_compare_raw(h, w.golden, w.candidate, w.rtol, w.atol, stats, hist, stream)
        else:
            peat.peat_compare_segmented_raw(h, w.golden, w.candidate, w.offsets, w.rtol, w.atol, stats, hist, stream)

    gc.collect()  # the oracle leg's garbage is not collected inside the timed batches
    for _ in range(3):
        call()
    est = events_ms(torch, stream, call, 3)
    # five batches of back-to-back calls (about 50 ms in all); the median batch
    # is the figure, so that one host stall (a segmented call waits on the host
    # for the previous call's staging copy) does not stand for the steady state
    per = int(min(1000, max(2, 10.0 / max(est, 1e-3))))
    batches = [events_ms(torch, stream, call, per) for _ in range(5)]
    ms = statistics.median(batches)
    nbytes = 2 * w.n * (4 if w.dtype == "f32" else 2)
    gbs = nbytes / (ms * 1e-3) / 1e9
    out = {"workload": WORKLOAD_NAMES[name], "element": w.dtype, "pairs": w.n, "segments": nseg,
           "algorithmic_bytes_per_call": nbytes,
           "hot": {"calls": 5 * per, "batches": 5, "us_per_call": ms * 1e3,
                   "us_per_call_batches": [round(b * 1e3, 1) for b in batches],
                   "pairs_per_s": w.n / (ms * 1e-3), "gbs": gbs,
                   "frac": gbs / peak, "l2": "back to back" + (" (inputs fit in L2: re-read from L2)"
                                                             if nbytes < 120e6 else " (inputs larger than L2)")}}
    if cold:
        flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
        times = []
        for i in range(30):
            flush.fill_(i & 255)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            call()
            e1.record(stream)
            torch.cuda.synchronize()
            times.append(e0.elapsed_time(e1))
        del flush
        cm = statistics.median(times)
        out["cold"] = {"calls": len(times), "us_per_call_median": cm * 1e3, "pairs_per_s": w.n / (cm * 1e-3),
                       "gbs": nbytes / (cm * 1e-3) / 1e9, "frac": nbytes / (cm * 1e-3) / 1e9 / peak,
                       "l2": "flushed before every call (512 MiB write, outside the timed call)"}
    if nseg > 1:
        mid = torch.cuda.Event(enable_timing=True)
        mid.record(stream)
        torch.cuda.synchronize()
        peat.peat_set_stage1_event(h, mid)
        s1, s2 = [], []
        try:
            for _ in range(20):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                call()
                e1.record(stream)
                torch.cuda.synchronize()
                s1.append(e0.elapsed_time(mid))
                s2.append(mid.elapsed_time(e1))
        finally:
            peat.peat_set_stage1_event(h, None)
        a, b = statistics.median(s1), statistics.median(s2)
        out["stage1_alone"] = {"us_stage1": a * 1e3, "us_finalize": b * 1e3, "us_total": (a + b) * 1e3,
                               "stage1_gbs": nbytes / (a * 1e-3) / 1e9, "stage1_frac": nbytes / (a * 1e-3) / 1e9 / peak,
                               "how": "events around each call and one the library records after the stage-1 "
                                      "launch (peat_set_stage1_event); medians of 20 calls"}
    del stats, hist
    return out


def c5_sweep(peat, h, stream, peak: float) -> dict:
    """Config 5 as specified: 64 successive step snapshots of the
    268,435,456-element bf16 tensor, generated beforehand (about 69 GB in
    HBM), compared back to back in one timed region; the per-step series and
    the cross-step trends (peat_trend) of mean |d| and max |d|."""
    import numpy as np
    import torch
    from paper_2609_13544_gb300 import workloads as W
    sweep = W.PlaybackSweep(device="cuda")
    n, S = sweep.n, 64
    G = torch.empty((S, n), dtype=torch.bfloat16, device="cuda")
    C = torch.empty((S, n), dtype=torch.bfloat16, device="cuda")
    for s in range(S):
        sweep.step(s, out_g=G[s], out_c=C[s])
    del sweep
    rtol = 2.0 ** -7
    stats = torch.empty(S * peat.STATS_BYTES, dtype=torch.uint8, device="cuda")
    hist = torch.empty(S * peat.HIST_BINS, dtype=torch.int64, device="cuda")

    def one(s):
        peat.peat_compare_raw(h, G[s], C[s], rtol, 0.0, stats[s * peat.STATS_BYTES:(s + 1) * peat.STATS_BYTES],
                              hist[s * peat.HIST_BINS:(s + 1) * peat.HIST_BINS], stream)

    for s in range(3):
        one(s)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(S):
        one(s)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    st = peat.stats_to_dicts(stats.cpu().numpy())
    del G, C, stats, hist
    torch.cuda.empty_cache()
    steps = list(range(S))
    mean_abs = [d["mean_abs"] for d in st]
    max_abs = [d["max_abs"] for d in st]
    nbytes = 2 * n * 2
    return {"workload": "playback sweep: steps 0..63 of a 268,435,456-element bf16 tensor, golden_s = x0 + s drift, "
                        "candidate_s = golden_s (1 + 1e-4 sqrt(s) z) rounded to bf16, rtol 2^-7",
            "steps": S, "pairs_per_step": n, "ms_total": ms, "us_per_step": ms * 1e3 / S,
            "pairs_per_s": S * n / (ms * 1e-3), "gbs": S * nbytes / (ms * 1e-3) / 1e9,
            "frac": S * nbytes / (ms * 1e-3) / 1e9 / peak,
            "step0_all_exact": st[0]["exact"] == n,
            "series": {"max_abs": max_abs, "mean_abs": mean_abs, "var_abs": [d["var_abs"] for d in st],
                       "non_exact": [d["n"] - d["exact"] for d in st], "mismatch": [d["mismatch"] for d in st],
                       "max_ulp": [d["max_ulp"] for d in st]},
            "trend_mean_abs": peat.peat_trend(steps, mean_abs), "trend_max_abs": peat.peat_trend(steps, max_abs),
            "note": "trend = least-squares slope of log score against log step over the steps with a nonzero "
                    "score (peat_trend); the injected noise grows like sqrt(s) but a bf16 candidate differs "
                    "only where it exceeds half a bf16 step, so mean |d| follows that Gaussian tail"}


# --------------------------------------------------------------------------- the CUDA path
def run_gpu(args) -> None:
    import numpy as np
    import torch

    import paper_2609_13544_gb300 as peat

    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    peat.load()
    w = make_workload(args.workload, "cuda")
    g, c = w.golden.to(dev), w.candidate.to(dev)
    nseg = 1 if w.offsets is None else len(w.offsets) - 1
    h = peat.Handle(local, max_segments=max(4096, nseg))
    stats = torch.empty(nseg * peat.STATS_BYTES, dtype=torch.uint8, device=dev)
    hist = torch.empty(nseg * peat.HIST_BINS, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        if w.offsets is None:
            peat.peat_compare_raw(h, g, c, w.rtol, w.atol, stats, hist, stream)
        else:
            peat.peat_compare_segmented_raw(h, g, c, w.offsets, w.rtol, w.atol, stats, hist, stream)

    # sanity before timing: counts add up
    step()
    torch.cuda.synchronize()
    st = peat.stats_to_dicts(stats.cpu().numpy())
    assert sum(sum(s["count"]) for s in st) == w.n, "counts do not add up to n"
    peaks = measured_peaks()
    peak = float(peaks.get("hbm_gbs", 6800.0))

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        torch.cuda.synchronize()

    # N = 1: the oracle leg first (the cpu_baseline of every config, and on
    # the same sample the parity of the CUDA path, before anything is timed),
    # then each config's own timings
    cpu, parity, configs = None, None, None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        cores = os.cpu_count() or 1
        configs = {}
        with make_pool(cores) as pool:
            for name in sorted(WORKLOAD_NAMES):
                wn = w if name == args.workload else make_workload(name, "cuda")
                r0 = oracle_sample(wn, pool, cores, min(wn.n, 50_000 * cores))[0]
                seconds = 15.0 if name == args.workload else 3.0  # oracle work per config (wall)
                rate, dt, done, off, ost, oh = oracle_sample(wn, pool, cores, int(max(1_000_000, r0 * seconds)))
                c_cpu = {"value": rate, "unit": "pairs/s", "cores": cores, "kind": "oracle",
                         "sample": f"first {done} pairs of {name} cut into {len(off) - 1} segments "
                                   f"(its own boundaries and {cores} equal chunks), {cores} processes, {dt:.1f} s wall"}
                c_par = parity_on_sample(peat, h, wn, off, ost, oh)
                del ost, oh
                blk = config_block(peat, h, name, wn, stream, peak, cold=name in ("c1", "c3"))
                blk["cpu_baseline"] = c_cpu
                blk["parity_before_timing"] = c_par
                blk["gpu_over_oracle"] = blk["hot"]["pairs_per_s"] / rate
                configs[name] = blk
                if name == args.workload:
                    cpu, parity = c_cpu, c_par
                del wn
                torch.cuda.empty_cache()

    # at least W warm-up steps, and at least 200 ms of them (the timed region
    # then starts in the steady state the sustained region below also sees)
    for _ in range(args.warmup):
        step()
    barrier()
    w0 = time.perf_counter()
    while time.perf_counter() - w0 < 0.2:
        for _ in range(20):
            step()
        barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    nvml = NvmlSampler(local)
    with (nvml if nvml.available else ClockSampler(local)) as clk:
        time.sleep(0.25)
        barrier()
        wall0 = time.perf_counter()
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        barrier()
        wall1 = time.perf_counter()
        wall = wall1 - wall0
        # a clock-covered region of at least a second: the same call repeated
        per = max(e0.elapsed_time(e1) / args.steps, 1e-3)
        sus_calls = int(max(args.steps, 1.5e3 / per))
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        sw0 = time.perf_counter()
        s0.record(stream)
        for _ in range(sus_calls):
            step()
        s1.record(stream)
        barrier()
        sw1 = time.perf_counter()
        time.sleep(0.25)
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    if nvml.available:
        clocks = nvml.summary(wall0, wall1)
        clocks_sus = nvml.summary(sw0, sw1)
    else:
        clocks = clocks_sus = clk.summary()
    ms_per_step = ms / args.steps
    value = whole_job_rate(w.n, world, args.steps, ms)
    bytes_per_step = 2 * w.n * (4 if w.dtype == "f32" else 2)
    gbs = bytes_per_step / (ms_per_step * 1e-3) / 1e9
    sus_ms = max_over_ranks(s0.elapsed_time(s1), dev) / sus_calls
    sustained = {"calls": sus_calls, "seconds": sus_ms * sus_calls * 1e-3, "us_per_call": sus_ms * 1e3,
                 "pairs_per_s": w.n / (sus_ms * 1e-3), "gbs": bytes_per_step / (sus_ms * 1e-3) / 1e9,
                 "frac": bytes_per_step / (sus_ms * 1e-3) / 1e9 / peak, "clocks": clocks_sus,
                 "us_x_sm_mhz": (sus_ms * 1e3 * clocks_sus["sm_mhz"]) if clocks_sus.get("sm_mhz") else None}
    if clocks.get("sm_mhz"):
        clocks["ms_per_step_x_sm_mhz"] = ms_per_step * clocks["sm_mhz"]
    sweep = None
    if rank == 0 and world == 1 and not args.no_sweep:
        sweep = c5_sweep(peat, h, stream, peak)

    # the mean of the top 10 % of the errors (Section IV-B-3) on the same
    # tensor: its own timing, reported beside the compare's line
    topk = None
    if w.offsets is None and not args.no_topk:
        tk_out = torch.empty(peat.TOPK_BYTES, dtype=torch.uint8, device=dev)
        for _ in range(3):
            peat.peat_topk_mean_raw(h, g, c, 1, 10, tk_out, stream)
        barrier()
        tk_calls = max(100, min(400, 5 * args.steps))
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(tk_calls):
            peat.peat_topk_mean_raw(h, g, c, 1, 10, tk_out, stream)
        t1.record(stream)
        barrier()
        tk_ms = max_over_ranks(t0.elapsed_time(t1), dev) / tk_calls
        r = np.frombuffer(tk_out.cpu().numpy().tobytes(), dtype=peat.TOPK_DTYPE)[0]
        read_gbs = bytes_per_step / (tk_ms * 1e-3) / 1e9
        topk = {"op": "peat_topk_mean, num/den = 1/10", "calls": tk_calls, "us_per_call": tk_ms * 1e3,
                "pairs_per_s": w.n / (tk_ms * 1e-3), "k": int(r["k"]), "exact": int(r["exact"]),
                "roofline": {"bound": "hbm", "achieved": read_gbs, "peak": peak, "unit": "GB/s",
                             "frac": read_gbs / peak, "algorithmic_bytes_per_call": bytes_per_step,
                             "note": "one read of both tensors (the counting pass); the last-digit pass reads "
                                     "them again unless the counting pass resolved it (16-bit operands whose "
                                     "window keys are multiples of 2^10 and exact), plus a sample and "
                                     "one-CTA selects"}}

    # the context statistics of the golden tensor(s) (Section IV-C-2): one read
    tstats = None
    if not args.no_topk:
        off = [0, w.n] if w.offsets is None else list(w.offsets)
        ts_out = torch.empty((len(off) - 1) * peat.TSTATS_BYTES, dtype=torch.uint8, device=dev)
        for _ in range(3):
            peat.peat_tensor_stats_raw(h, g, off, ts_out, stream)
        barrier()
        ts_calls = max(100, min(400, 5 * args.steps))
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(ts_calls):
            peat.peat_tensor_stats_raw(h, g, off, ts_out, stream)
        t1.record(stream)
        barrier()
        ts_ms = max_over_ranks(t0.elapsed_time(t1), dev) / ts_calls
        one = bytes_per_step // 2
        ts_gbs = one / (ts_ms * 1e-3) / 1e9
        tstats = {"op": "peat_tensor_stats of the golden tensor(s)", "calls": ts_calls, "segments": len(off) - 1,
                  "us_per_call": ts_ms * 1e3, "elements_per_s": w.n / (ts_ms * 1e-3),
                  "roofline": {"bound": "hbm", "achieved": ts_gbs, "peak": peak, "unit": "GB/s",
                               "frac": ts_gbs / peak, "algorithmic_bytes_per_call": one,
                               "note": "one read of the tensor; stage 1 plus a per-segment finalize"}}

    # isclose pass counts over an 8 x 8 tolerance grid (Section III-A, Fig. 5): one read of both tensors
    isc = None
    if not args.no_topk:
        rts = [0.0, 1e-5, 1e-4, 1e-3, 2.0 ** -7, 1e-2, 0.1, 1.0]
        ats = [0.0, 1e-8, 1e-6, 1e-4, 1e-2, 1.0, 1e3, 1e30]
        ic_out = torch.empty(64, dtype=torch.int64, device=dev)
        for _ in range(3):
            peat.peat_isclose_grid_raw(h, g, c, rts, ats, ic_out, stream)
        barrier()
        ic_calls = max(10, min(50, args.steps // 100))
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(ic_calls):
            peat.peat_isclose_grid_raw(h, g, c, rts, ats, ic_out, stream)
        t1.record(stream)
        barrier()
        ic_ms = max_over_ranks(t0.elapsed_time(t1), dev) / ic_calls
        ic_gbs = bytes_per_step / (ic_ms * 1e-3) / 1e9
        isc = {"op": "peat_isclose_grid, 8 rtols x 8 atols", "calls": ic_calls, "us_per_call": ic_ms * 1e3,
               "pairs_per_s": w.n / (ic_ms * 1e-3),
               "roofline": {"bound": "alu", "achieved": ic_gbs, "peak": peak, "unit": "GB/s", "frac": ic_gbs / peak,
                            "algorithmic_bytes_per_call": bytes_per_step,
                            "note": "one read of both tensors; 64 exact tolerance decisions per differing pair"}}

    # fused inject + compare (Alg. 1's Inject and Compare in one read of the golden): the
    # candidate g (1 + 1e-3 z) generated in the kernel, against the injector writing it
    # followed by the compare reading both
    fused = None
    if w.offsets is None and not args.no_topk:
        scratch = torch.empty_like(g)
        cnt = torch.zeros(1, dtype=torch.int64, device=dev)
        fu_calls = max(10, min(100, args.steps // 50))

        def timed(fn):
            for _ in range(3):
                fn()
            barrier()
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            for _ in range(fu_calls):
                fn()
            t1.record(stream)
            barrier()
            return max_over_ranks(t0.elapsed_time(t1), dev) / fu_calls

        per_model = {}
        for name, x in (("rel_gauss", 1e-3), ("bias", 1e-3)):
            models = [peat.inject_model(name, x=x)]
            ms_inj = timed(lambda: peat.peat_pseudo_error_inject_raw(h, scratch, g, models, 9, cnt, stream))
            ms_cmp = timed(lambda: peat.peat_compare_raw(h, g, scratch, w.rtol, w.atol, stats, hist, stream))
            ms_fu = timed(lambda: peat.peat_inject_compare_raw(h, g, models, 9, w.rtol, w.atol, stats, hist, stream))
            per_model[f"{name} {x:g}"] = {"fused_us": ms_fu * 1e3, "inject_us": ms_inj * 1e3,
                                          "compare_us": ms_cmp * 1e3, "speedup": (ms_inj + ms_cmp) / ms_fu}
        head = per_model["rel_gauss 0.001"]
        one = bytes_per_step // 2
        fu_gbs = one / (head["fused_us"] * 1e-6) / 1e9
        fused = {"op": "peat_inject_compare on the golden, against peat_pseudo_error_inject into a scratch "
                       "tensor followed by peat_compare", "calls": fu_calls,
                 "us_per_call": head["fused_us"], "pairs_per_s": w.n / (head["fused_us"] * 1e-6),
                 "per_model": per_model,
                 "roofline": {"bound": "alu", "achieved": fu_gbs, "peak": peak, "unit": "GB/s",
                              "frac": fu_gbs / peak, "algorithmic_bytes_per_call": one,
                              "note": "rel_gauss: one read of the golden; per four elements one Philox4x32-10 "
                                      "draw and two Box-Muller pairs, then the compare"}}
        del scratch

    # the 8-bit formats (OCP FP8): the golden's values rounded to E4M3 / E5M2 against the same
    # values with relative noise 2^-4, rounded the same way; one read of both 1-byte tensors
    fp8 = None
    if w.offsets is None and not args.no_topk:
        fp8 = {}
        gen = torch.Generator(device=dev)
        gen.manual_seed(17)
        x = g.float()
        y = x * (1.0 + 0.0625 * torch.randn(x.shape, generator=gen, device=dev))
        for name, tdt in (("e4m3", torch.float8_e4m3fn), ("e5m2", torch.float8_e5m2)):
            g8, c8 = x.to(tdt), y.to(tdt)
            for _ in range(3):
                peat.peat_compare_raw(h, g8, c8, 0.125, 0.0, stats, hist, stream)
            barrier()
            calls = max(10, min(100, args.steps // 50))
            t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            for _ in range(calls):
                peat.peat_compare_raw(h, g8, c8, 0.125, 0.0, stats, hist, stream)
            t1.record(stream)
            barrier()
            ms = max_over_ranks(t0.elapsed_time(t1), dev) / calls
            gbs8 = 2 * w.n / (ms * 1e-3) / 1e9
            fp8[name] = {"us_per_call": ms * 1e3, "pairs_per_s": w.n / (ms * 1e-3),
                         "roofline": {"bound": "alu", "achieved": gbs8, "peak": peak, "unit": "GB/s",
                                      "frac": gbs8 / peak, "algorithmic_bytes_per_call": 2 * w.n}}
            del g8, c8
        del x, y
        fp8 = {"op": "peat_compare on 8-bit golden and candidate (rtol 1/8)", "calls": calls, **fp8}

    # binary64 (Fig. 5's FP32-FP64 pairs): the golden's values plus noise 1e-3 in binary64, against
    # their float32 rounding widened back to binary64; one read of both 8-byte tensors
    f64 = None
    if w.offsets is None and not args.no_topk:
        gen = torch.Generator(device=dev)
        gen.manual_seed(19)
        g64 = g.double() + 1e-3 * torch.randn(g.shape, generator=gen, device=dev, dtype=torch.float64)
        c64 = g64.float().double()
        for _ in range(3):
            peat.peat_compare_raw(h, g64, c64, 1e-7, 0.0, stats, hist, stream)
        barrier()
        calls = max(5, min(20, args.steps // 200))
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(calls):
            peat.peat_compare_raw(h, g64, c64, 1e-7, 0.0, stats, hist, stream)
        t1.record(stream)
        barrier()
        ms = max_over_ranks(t0.elapsed_time(t1), dev) / calls
        gbs64 = 16 * w.n / (ms * 1e-3) / 1e9
        f64 = {"op": "peat_compare on binary64 golden and its float32 rounding (rtol 1e-7)", "calls": calls,
               "us_per_call": ms * 1e3, "pairs_per_s": w.n / (ms * 1e-3),
               "roofline": {"bound": "alu", "achieved": gbs64, "peak": peak, "unit": "GB/s", "frac": gbs64 / peak,
                            "algorithmic_bytes_per_call": 16 * w.n,
                            "note": "FP64 TwoSum per pair and the three sums as digit atomics in shared memory"}}
        del g64, c64

    # end to end through the C ABI with host buffers: every step copies both
    # tensors from pinned host memory, compares them and reads the stats and
    # histograms back.  Two device buffer sets: step i's copies (copy stream)
    # overlap step i-1's compare (compute stream); events order the reuse.
    e2e = None
    if rank == 0 or world > 1:
        gh = torch.empty_like(g, device="cpu").pin_memory()
        ch = torch.empty_like(c, device="cpu").pin_memory()
        gh.copy_(g)
        ch.copy_(c)
        sh = torch.empty_like(stats, device="cpu").pin_memory()
        hh = torch.empty_like(hist, device="cpu").pin_memory()
        bufs = [(g, c), (torch.empty_like(g), torch.empty_like(c))]
        copy_stream = torch.cuda.Stream(dev)
        copied = [torch.cuda.Event(), torch.cuda.Event()]
        freed = [torch.cuda.Event(), torch.cuda.Event()]
        for ev in freed:
            ev.record(stream)
        e2e_steps = max(3, min(args.steps, 50))

        def e2e_step(i):
            k = i & 1
            bg, bc = bufs[k]
            copy_stream.wait_event(freed[k])  # the compare that last read this buffer set is done
            with torch.cuda.stream(copy_stream):
                bg.copy_(gh, non_blocking=True)
                bc.copy_(ch, non_blocking=True)
                copied[k].record(copy_stream)
            stream.wait_event(copied[k])
            if w.offsets is None:
                peat.peat_compare_raw(h, bg, bc, w.rtol, w.atol, stats, hist, stream)
            else:
                peat.peat_compare_segmented_raw(h, bg, bc, w.offsets, w.rtol, w.atol, stats, hist, stream)
            freed[k].record(stream)
            sh.copy_(stats, non_blocking=True)
            hh.copy_(hist, non_blocking=True)

        for i in range(2):
            e2e_step(i)
        barrier()
        f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        f0.record(stream)
        copy_stream.wait_event(f0)
        for i in range(e2e_steps):
            e2e_step(i)
        f1.record(stream)
        barrier()
        ems = max_over_ranks(f0.elapsed_time(f1), dev)
        e2e = {"value": whole_job_rate(w.n, world, e2e_steps, ems), "unit": "pairs/s",
               "h2d_bytes_per_step": bytes_per_step, "d2h_bytes_per_step": int(stats.numel() + hist.numel() * 8),
               "ms_per_step": ems / e2e_steps,
               "note": "pinned H2D of both tensors every step on a copy stream, overlapped with the previous "
                       "step's compare (two buffer sets); stats and histograms read back every step"}
        del bufs

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "pairs/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32+int (exact)", "data": "synthetic",
            "config": {"workload": WORKLOAD_NAMES[args.workload], "element": w.dtype, "pairs": w.n,
                       "segments": nseg, "l2": "inputs larger than L2 (no flush)" if bytes_per_step > 135e6
                       else "inputs smaller than L2: steps re-read from L2", "parallelism": f"replicas x{world}"},
            "hbm_gbs": gbs, "frac_of_8tbs": gbs / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s", "frac": gbs / peak,
                         "traffic": recorded_traffic(args.workload),
                         "kernel": ("compare_stage1<%s>, the one launch of each call (finalization in the same "
                                    "kernel), event-timed on the launch stream" % w.dtype) if nseg == 1 else
                                   ("compare_stage1<%s> + compare_finalize per call, event-timed together on the "
                                    "launch stream" % w.dtype),
                         "algorithmic_bytes_per_launch": bytes_per_step,
                         "peak_source": "MEASURED_PEAKS.json hbm_gbs (copy)" if not peaks.get("fallback")
                         else "fallback 6.8 TB/s"},
            "e2e": e2e, "cpu_baseline": cpu, "gpu_launches": (1 if nseg == 1 else 2) * args.steps, "clocks": clocks,
            "parity_before_timing": parity, "sustained": sustained, "configs": configs, "c5_sweep": sweep,
            "next_rows": {"f1_top10_mean": topk, "f2_fused_inject_compare": fused, "f3_context_stats": tstats,
                          "f4_isclose_grid": isc, "f4_fp8_compare": fp8, "f4_f64_compare": f64},
            "wall_s_timed": wall,
        }
        print(json.dumps(line), flush=True)
    h.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="c2", choices=sorted(WORKLOAD_NAMES))
    ap.add_argument("--impl", default="peat", choices=["peat", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true", help="skip the 64-step config-5 sweep")
    ap.add_argument("--no-topk", action="store_true",
                    help="skip the timings of the next rows (top-10 %% mean, fused inject + compare, "
                         "context statistics, isclose grid)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.steps is None:
        args.steps = {"c1": 20000, "c2": 20000, "c3": 20000, "c4": 3000, "c5": 4000}[args.workload]
        if args.impl == "reference":
            args.steps = 10
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
