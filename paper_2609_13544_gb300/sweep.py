"""Playback sweeps with checkpoint/resume.

Alg. 1 of the paper replays the recorded epochs one after another and runs
its Err step (the error signature of the replayed output against the
golden) once per epoch; Section IV-C-1 then reads each layer's scores across
the epochs.  ``playback_sweep`` runs that loop over step snapshots: for
every step it obtains the (golden, candidate) pair, computes its signature
with ``peat_compare`` (the library's CUDA path), and returns the per-step
series of the scores and their cross-step trends (``peat_trend``).

With ``record_dir`` each step's record is written to
``record_dir/step_NNNNNN.json`` as soon as the step is done (written to a
temporary file and renamed, so a record is either complete or absent), and a
rerun with the same directory skips every step whose record is there and
matches the sweep's settings: an interrupted sweep resumes where it stopped.
"""
from __future__ import annotations

import json
import os
from pathlib import Path
from typing import Callable, Iterable, Optional

RECORD_VERSION = 1


def _fingerprint(rtol: float, atol: float, tag: str) -> dict:
    return {"version": RECORD_VERSION, "rtol": float(rtol), "atol": float(atol), "tag": tag}


def _load_record(path: Path, fp: dict) -> Optional[dict]:
    """A step's record if it is complete and was made with the same settings."""
    try:
        rec = json.loads(path.read_text())
    except (OSError, ValueError):
        return None
    if not isinstance(rec, dict) or rec.get("fingerprint") != fp or "stats" not in rec or "hist" not in rec:
        return None
    return rec


def _write_record(path: Path, rec: dict) -> None:
    tmp = path.with_name(path.name + f".tmp{os.getpid()}")
    tmp.write_text(json.dumps(rec))
    os.replace(tmp, path)


def playback_sweep(h, step_fn: Callable[[int], tuple], steps: Iterable[int], rtol: float, atol: float = 0.0,
                   record_dir=None, tag: str = "", compare_fn=None) -> dict:
    """The error signature of every step of a playback sweep.

    step_fn(s) returns the step's (golden, candidate) device tensors;
    compare_fn(h, golden, candidate, rtol, atol) -> (stats dict, hist) is
    ``peat_compare`` unless given.  ``tag`` names the sweep in its records
    (a record of another tag, rtol or atol is recomputed, not reused).
    Returns {"steps", "records" (per step: stats and hist as lists, and
    whether it was resumed), "series" (max_abs, mean_abs, var_abs,
    non_exact, mismatch, max_ulp), "trend_mean_abs", "trend_max_abs",
    "computed", "resumed"}."""
    import numpy as np

    from . import peat_compare, peat_trend
    compare = compare_fn or peat_compare
    fp = _fingerprint(rtol, atol, tag)
    rdir = Path(record_dir) if record_dir is not None else None
    if rdir is not None:
        rdir.mkdir(parents=True, exist_ok=True)
    steps = [int(s) for s in steps]
    records, computed, resumed = [], 0, 0
    for s in steps:
        path = rdir / f"step_{s:06d}.json" if rdir is not None else None
        rec = _load_record(path, fp) if path is not None and path.exists() else None
        if rec is not None and rec.get("step") == s:
            rec["resumed"] = True
            resumed += 1
        else:
            g, c = step_fn(s)
            st, hist = compare(h, g, c, rtol, atol)
            rec = {"step": s, "fingerprint": fp, "stats": st,
                   "hist": np.asarray(hist, dtype=np.uint64).astype(int).tolist()}
            if path is not None:
                _write_record(path, rec)
            rec = dict(rec, resumed=False)
            computed += 1
        records.append(rec)
    stats = [r["stats"] for r in records]
    series = {k: [st[k] for st in stats] for k in ("max_abs", "mean_abs", "var_abs", "mismatch", "max_ulp")}
    series["non_exact"] = [st["n"] - st["exact"] for st in stats]
    return {"steps": steps, "records": records, "series": series,
            "trend_mean_abs": peat_trend(steps, series["mean_abs"]),
            "trend_max_abs": peat_trend(steps, series["max_abs"]),
            "computed": computed, "resumed": resumed}
