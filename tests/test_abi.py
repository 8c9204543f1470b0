"""The C-ABI library builds, loads and exports every symbol include/peat.h declares (CPU only)."""
import ctypes
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def declared_functions():
    text = (ROOT / "include" / "peat.h").read_text()
    return sorted(set(re.findall(r"^(?:peat_status_t|const char\*|void)\s+(peat_\w+)\s*\(", text, re.M)))


def test_header_declares_the_boundary():
    assert declared_functions() == sorted([
        "peat_compare", "peat_compare_noalloc", "peat_compare_segmented", "peat_inject_compare", "peat_last_error",
        "peat_isclose_grid", "peat_mean_std", "peat_pseudo_error_inject", "peat_signature_create",
        "peat_signature_destroy",
        "peat_spearman", "peat_tensor_stats", "peat_test_noalloc_expire_waits", "peat_topk_mean"])


def test_library_builds_and_exports_every_declared_symbol():
    from paper_2609_13544_gb300 import buildlib
    lib = buildlib.build()
    L = ctypes.CDLL(str(lib))
    for name in declared_functions():
        assert hasattr(L, name), name


def test_binding_names_match_the_abi():
    import paper_2609_13544_gb300 as peat
    for name in declared_functions():
        assert hasattr(peat, name), name
    assert peat.STATS_DTYPE.itemsize == 144
    assert peat.TOPK_DTYPE.itemsize == 48
    assert peat.TSTATS_DTYPE.itemsize == 80


def test_last_error_without_handle_is_empty_string():
    import paper_2609_13544_gb300 as peat
    peat.build()
    assert isinstance(peat.peat_last_error(None), str)


def test_stats_layout_matches_oracle():
    import oracle
    import paper_2609_13544_gb300 as peat
    assert ctypes.sizeof(oracle.Stats) == peat.STATS_DTYPE.itemsize
    assert [f for f, _ in oracle.Stats._fields_] == list(peat.STATS_DTYPE.names)
