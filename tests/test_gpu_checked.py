"""The checked build (libpeat_checked.so, -DPEAT_CHECKED): the compare kernels
assert their indices and ranges into the library's status word instead of
trusting them.  In a child process (so the suite's own library stays the one
loaded here) the checked library runs a mixture of one-tensor, misaligned
and segmented compares of all three operand widths; every result must equal
the oracle's and no assertion may fire (the next call returns PEAT_OK, not
PEAT_ERR_INTERNAL)."""
import subprocess
import sys
from pathlib import Path

import pytest

pytestmark = pytest.mark.gpu
ROOT = Path(__file__).resolve().parents[1]

CHILD = r'''
import sys
sys.path.insert(0, sys.argv[1]); sys.path.insert(0, sys.argv[1] + "/tests")
import numpy as np, torch
import oracle
import paper_2609_13544_gb300 as peat
from paper_2609_13544_gb300 import buildlib
from parity_util import random_pairs, noise_pairs, to_device, assert_stats_equal, assert_hist_equal
lib = buildlib.build(checked=True)
peat.load(lib)
assert peat.load()._name.endswith("libpeat_checked.so")
h = peat.Handle(0, max_segments=64)
for dt in ("f32", "f16", "bf16"):
    for n, off in ((1, 0), (4099, 1), (300_001, 0), (1_000_003, 3)):
        gb, cb = random_pairs(dt, n, seed=n + len(dt))
        st, hist = peat.peat_compare(h, to_device(gb, dt, off), to_device(cb, dt), 1e-3, 0.0)
        ost, oh = oracle.compare(gb, cb, dt, 1e-3, 0.0)
        assert_stats_equal(st, ost, f"{dt} n={n}")
        assert_hist_equal(hist, oh, f"{dt} n={n}")
    gb, cb = noise_pairs(dt, 2_000_000, seed=7)
    offs = [0, 5, 70_000, 70_001, 1_000_000, 2_000_000]
    st, hist = peat.peat_compare_segmented(h, to_device(gb, dt), to_device(cb, dt), offs, 1e-3, 0.0)
    ost, oh = oracle.compare_segmented(gb, cb, offs, dt, 1e-3, 0.0)
    for s in range(len(ost)):
        assert_stats_equal(st[s], ost[s], f"{dt} seg {s}")
    assert_hist_equal(hist, oh, f"{dt} segmented")
torch.cuda.synchronize()
x = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
peat.peat_compare(h, x, x, 1e-3, 0.0)  # raises PEAT_ERR_INTERNAL if any assertion fired
h.close()
print("checked build ok")
'''


def test_checked_build_matches_the_oracle_and_asserts_nothing():
    r = subprocess.run([sys.executable, "-c", CHILD, str(ROOT)], capture_output=True, text=True, timeout=1200)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "checked build ok" in r.stdout
