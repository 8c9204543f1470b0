"""Build the oracle's shared library with gcc (test infrastructure only).

The oracle is plain C: it is compiled without contraction of a*b+c into
fused multiply-adds (-ffp-contract=off) and without fast-math, so every
binary64 and binary32 operation rounds once, as written.
"""
import os
import subprocess
from pathlib import Path

HERE = Path(__file__).resolve().parent
SRC = HERE / "peat_oracle.c"
HDR = HERE / "peat_oracle.h"
OUT_DIR = HERE / "_build"
LIB = OUT_DIR / "libpeat_oracle.so"

CFLAGS = ["-O2", "-std=gnu11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
          "-Wall", "-Wextra", "-Wno-unused-parameter"]


def build(force: bool = False) -> Path:
    """Compile oracle/peat_oracle.c into oracle/_build/libpeat_oracle.so."""
    OUT_DIR.mkdir(exist_ok=True)
    if (not force and LIB.exists()
            and LIB.stat().st_mtime >= max(SRC.stat().st_mtime, HDR.stat().st_mtime)):
        return LIB
    tmp = OUT_DIR / f"libpeat_oracle.{os.getpid()}.so"
    cmd = [os.environ.get("CC", "gcc"), *CFLAGS, "-o", str(tmp), str(SRC), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True))
