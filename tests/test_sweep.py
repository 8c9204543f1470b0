"""Checkpoint/resume of a playback sweep (paper_2609_13544_gb300.sweep): host
logic, run on the CPU with a stand-in for the compare (the CUDA path itself
is covered by the gpu tests); the trends come from the library's host
function peat_trend."""
import json
import math

import numpy as np
import pytest


@pytest.fixture(scope="module")
def peat_host():
    import paper_2609_13544_gb300 as peat
    from paper_2609_13544_gb300 import buildlib
    buildlib.build()
    peat.load()
    return peat


class FakeCompare:
    """Deterministic signatures: step s has mean |d| = 1e-4 sqrt(s + 1)."""

    def __init__(self, fail_at=None):
        self.calls = []
        self.fail_at = fail_at

    def __call__(self, h, g, c, rtol, atol):
        s = g
        if self.fail_at is not None and s == self.fail_at:
            raise RuntimeError("interrupted")
        self.calls.append(s)
        st = {"n": 1000, "exact": 1000 - 10 * s, "mismatch": s, "max_abs": 1e-3 * (s + 1), "max_ulp": s,
              "mean_abs": 1e-4 * math.sqrt(s + 1), "var_abs": 1e-9 * (s + 1), "count": [0, 0, 0, 0, 0]}
        hist = np.zeros((2, 64), np.uint64)
        hist[0, 0] = st["exact"]
        return st, hist


def step_fn(s):
    return s, s  # the stand-in compare receives the step number


def test_sweep_records_and_resumes(peat_host, tmp_path):
    from paper_2609_13544_gb300.sweep import playback_sweep
    steps = list(range(8))
    fake = FakeCompare()
    r1 = playback_sweep(None, step_fn, steps, 2.0 ** -7, record_dir=tmp_path, tag="t", compare_fn=fake)
    assert r1["computed"] == 8 and r1["resumed"] == 0 and fake.calls == steps
    assert sorted(p.name for p in tmp_path.iterdir()) == [f"step_{s:06d}.json" for s in steps]
    # slope of log mean |d| against log step: 1/2 for sqrt(s + 1) at s + 1 -- here against s, so
    # compare with the library trend of the same series instead
    want = peat_host.peat_trend(steps, [1e-4 * math.sqrt(s + 1) for s in steps])
    assert r1["trend_mean_abs"] == want
    # a rerun reads every record and computes nothing
    fake2 = FakeCompare()
    r2 = playback_sweep(None, step_fn, steps, 2.0 ** -7, record_dir=tmp_path, tag="t", compare_fn=fake2)
    assert fake2.calls == [] and r2["resumed"] == 8 and r2["series"] == r1["series"]
    assert [r["hist"] for r in r2["records"]] == [r["hist"] for r in r1["records"]]
    # a missing and a truncated record are recomputed, the others reused
    (tmp_path / "step_000003.json").unlink()
    p5 = tmp_path / "step_000005.json"
    p5.write_text(p5.read_text()[:20])
    fake3 = FakeCompare()
    r3 = playback_sweep(None, step_fn, steps, 2.0 ** -7, record_dir=tmp_path, tag="t", compare_fn=fake3)
    assert fake3.calls == [3, 5] and r3["series"] == r1["series"]
    # other settings (rtol, or another sweep's tag) never reuse a record
    fake4 = FakeCompare()
    playback_sweep(None, step_fn, steps, 1e-3, record_dir=tmp_path, tag="t", compare_fn=fake4)
    assert fake4.calls == steps
    fake5 = FakeCompare()
    playback_sweep(None, step_fn, steps, 1e-3, record_dir=tmp_path, tag="other", compare_fn=fake5)
    assert fake5.calls == steps


def test_interrupted_sweep_resumes_where_it_stopped(peat_host, tmp_path):
    from paper_2609_13544_gb300.sweep import playback_sweep
    steps = list(range(10))
    with pytest.raises(RuntimeError):
        playback_sweep(None, step_fn, steps, 2.0 ** -7, record_dir=tmp_path, compare_fn=FakeCompare(fail_at=6))
    assert sorted(p.name for p in tmp_path.iterdir()) == [f"step_{s:06d}.json" for s in range(6)]
    fake = FakeCompare()
    r = playback_sweep(None, step_fn, steps, 2.0 ** -7, record_dir=tmp_path, compare_fn=fake)
    assert fake.calls == [6, 7, 8, 9] and r["computed"] == 4 and r["resumed"] == 6
    rec = json.loads((tmp_path / "step_000009.json").read_text())
    assert rec["step"] == 9 and rec["stats"]["mismatch"] == 9
    # no temporary files are left behind
    assert not [p for p in tmp_path.iterdir() if ".tmp" in p.name]


def test_sweep_without_records(peat_host):
    from paper_2609_13544_gb300.sweep import playback_sweep
    fake = FakeCompare()
    r = playback_sweep(None, step_fn, [0, 2, 4], 2.0 ** -7, compare_fn=fake)
    assert fake.calls == [0, 2, 4] and r["computed"] == 3 and r["series"]["mismatch"] == [0, 2, 4]
