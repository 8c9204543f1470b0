"""Compile libpeat.so (the CUDA library behind include/peat.h) for sm_103a.

Each translation unit is compiled in parallel with nvcc, then linked into
paper_2609_13544_gb300/_build/libpeat.so.  No CMake; a rebuild happens when
any source or header is newer than the library.  build(checked=True) makes
libpeat_checked.so instead: the same sources with -DPEAT_CHECKED, whose
kernels assert indices and ranges into the library's status word.
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
CSRC = PKG / "csrc"
OUT_DIR = PKG / "_build"
LIB = OUT_DIR / "libpeat.so"
LIB_CHECKED = OUT_DIR / "libpeat_checked.so"
SOURCES = ["compare.cu", "compare8.cu", "compare64.cu", "topk.cu", "tstats.cu", "isclose.cu", "isclose64.cu", "inject.cu", "peat_api.cpp"]
HEADERS = [CSRC / "peat_internal.h", CSRC / "exact.cuh", CSRC / "meanvar.cuh", CSRC / "inject_models.cuh", CSRC / "tol_exact.cuh", CSRC / "exact64.cuh",
           ROOT / "include" / "peat.h"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              f"-I{ROOT / 'include'}", f"-I{CSRC}"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and Path(cand).exists():
            return cand
    raise RuntimeError("nvcc not found: the CUDA library cannot be built")


def _stale(lib: Path) -> bool:
    if not lib.exists():
        return True
    t = lib.stat().st_mtime
    deps = [CSRC / s for s in SOURCES] + HEADERS + [Path(__file__)]
    return any(d.stat().st_mtime > t for d in deps)


def build(force: bool = False, verbose: bool = False, checked: bool = False) -> Path:
    out = LIB_CHECKED if checked else LIB
    if not force and not _stale(out):
        return out
    OUT_DIR.mkdir(exist_ok=True)
    nv = nvcc()
    tag = os.getpid()

    def compile_one(src: str) -> Path:
        obj = OUT_DIR / f"{Path(src).stem}.{tag}{'.checked' if checked else ''}.o"
        lang = ["-x", "cu"] if src.endswith(".cpp") else []
        cmd = [nv, *ARCH, *NVCC_FLAGS, *(["-DPEAT_CHECKED"] if checked else []), *lang, "-c", str(CSRC / src),
               "-o", str(obj)]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and r.stderr:
            print(r.stderr)
        return obj

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        futs = [ex.submit(compile_one, src) for src in SOURCES]
    try:
        objs = [f.result() for f in futs]
    except Exception:
        for src in SOURCES:  # no objects of a failed build are left behind
            (OUT_DIR / f"{Path(src).stem}.{tag}{'.checked' if checked else ''}.o").unlink(missing_ok=True)
        raise
    tmp = OUT_DIR / f"{out.stem}.{tag}.so"
    cmd = [nv, *ARCH, "-shared", "-o", str(tmp), *map(str, objs), "-lcudart"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    for o in objs:
        o.unlink(missing_ok=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    import sys
    print(build(force=True, verbose="-v" in sys.argv))
