"""Lays out tests/golden/hand_cases.json.

Every expected value in this file was worked out by hand from the
definitions (Section IV-B-3: the error is the absolute difference of golden
and faulty values; the relative error, ULP distance, classes and bins as
read for this library), using IEEE 754 bit patterns.  Nothing here calls the
oracle or the CUDA library.  Run: python tests/golden/make_hand_cases.py
"""
import json
from pathlib import Path

ONE = {"f32": "0x3f800000", "f16": "0x3c00", "bf16": "0x3f80"}
NEXT1 = {"f32": "0x3f800001", "f16": "0x3c01", "bf16": "0x3f81"}
MONE = {"f32": "0xbf800000", "f16": "0xbc00", "bf16": "0xbf80"}
PZ = {"f32": "0x0", "f16": "0x0", "bf16": "0x0"}
NZ = {"f32": "0x80000000", "f16": "0x8000", "bf16": "0x8000"}
NAN = {"f32": "0x7fc00000", "f16": "0x7e00", "bf16": "0x7fc0"}
INF = {"f32": "0x7f800000", "f16": "0x7c00", "bf16": "0x7f80"}
NINF = {"f32": "0xff800000", "f16": "0xfc00", "bf16": "0xff80"}
MAX = {"f32": "0x7f7fffff", "f16": "0x7bff", "bf16": "0x7f7f"}
TWO = {"f32": "0x40000000", "f16": "0x4000", "bf16": "0x4000"}
ONE_P7 = {"f32": "0x3f810000", "f16": "0x3c08", "bf16": "0x3f81"}  # 1 + 2^-7
BIG = {"f32": "0x49800000", "f16": "0x7bff", "bf16": "0x4980"}  # 2^20 (fp16: 65504)
KEY1 = {"f32": 1065353216, "f16": 15360, "bf16": 16256}  # key(1.0) = bit pattern of 1.0
KEYINF = {"f32": 2139095040, "f16": 31744, "bf16": 32640}
EPSBIN = {"f32": 25, "f16": 38, "bf16": 41}  # rel = 2^-23, 2^-10, 2^-7 -> bin k + 48
U21 = {"f32": 8388608, "f16": 1024, "bf16": 128}  # key(2) - key(1): one binade of steps
UP7 = {"f32": 65536, "f16": 8, "bf16": 1}  # steps from 1 to 1 + 2^-7

SEC = ("Section IV-B-3 (error = |golden - faulty|); relative error, ULP distance, classes "
       "and bins as read for this library")


def main():
    cases = []

    def add(dt, g, c, cls, rb, ub, u, why, rtol=0.0, atol=0.0):
        cases.append({"dtype": dt, "g": g, "c": c, "rtol": rtol, "atol": atol, "class": cls,
                      "relbin": rb, "ulpbin": ub, "u": u, "why": why})

    for dt in ("f32", "f16", "bf16"):
        add(dt, ONE[dt], ONE[dt], "exact", 0, 0, 0, "equal values")
        add(dt, PZ[dt], NZ[dt], "exact", 0, 0, 0, "+0 and -0 are numerically equal; both keys are 0")
        add(dt, ONE[dt], NEXT1[dt], "mismatch", EPSBIN[dt], 1, 1, "one step above 1: rel = 2^-(p-1)")
        add(dt, ONE[dt], MONE[dt], "sign_flip", 49, 63, 2 * KEY1[dt], "|d| = 2, rel = 2 -> k = 1; signs differ, both nonzero")
        add(dt, PZ[dt], ONE[dt], "mismatch", 63, 63, KEY1[dt], "g = 0 < a: rel = +inf, bin 63")
        add(dt, NAN[dt], NAN[dt], "exact", 0, 0, None, "both NaN are equal non-finite; no ULP distance")
        add(dt, NAN[dt], ONE[dt], "nan_inf_asym", 63, 63, None, "NaN against a number")
        add(dt, INF[dt], MAX[dt], "nan_inf_asym", 63, 1, 1, "+Inf sits one key step past the largest finite value")
        add(dt, TWO[dt], ONE[dt], "mismatch", 47, 63, U21[dt], "rel = 1/2 -> k = -1")
        add(dt, ONE[dt], TWO[dt], "mismatch", 48, 63, U21[dt], "rel = 1 -> k = 0")
        add(dt, "0x1", "0x2", "mismatch", 48, 1, 1, "smallest subnormal vs twice it: rel = 1")
        add(dt, ONE[dt], ONE_P7[dt], "within_tol", 41, min(UP7[dt], 63), UP7[dt],
            "a = rtol*|g| exactly: the test is inclusive", rtol=2.0 ** -7)
        add(dt, ONE[dt], ONE_P7[dt], "mismatch", 41, min(UP7[dt], 63), UP7[dt],
            "rtol one float32 step below 2^-7", rtol=0.0078124995343387127)
        add(dt, ONE[dt], ONE_P7[dt], "within_tol", 41, min(UP7[dt], 63), UP7[dt], "a = atol exactly", atol=2.0 ** -7)
        add(dt, ONE[dt], MONE[dt], "within_tol", 49, 63, 2 * KEY1[dt], "tolerance precedes sign flip", atol=2.0)
        add(dt, INF[dt], NINF[dt], "nan_inf_asym", 63, 63, 2 * KEYINF[dt], "+Inf vs -Inf is asymmetric, not a sign flip")
        add(dt, INF[dt], INF[dt], "exact", 0, 0, 0, "equal infinities")
        add(dt, NZ[dt], ONE[dt], "mismatch", 63, 63, KEY1[dt], "g = -0: no sign flip when g = 0")
        add(dt, ONE[dt], NZ[dt], "mismatch", 48, 63, KEY1[dt], "c = -0: no sign flip when c = 0; rel = 1")
        add(dt, ONE[dt], PZ[dt], "within_tol", 48, 63, KEY1[dt], "a = 1 <= rtol*|g| with rtol = 1", rtol=1.0)
        add(dt, ONE[dt], BIG[dt], "mismatch", 62, 63, None, "rel >= 2^15 clamps to bin 62")
    add("f16", "0x3c00", "0x3c3e", "mismatch", 43, 62, 62, "u = 62 stays in bin 62; rel = 62/1024 -> k = -5")
    add("f16", "0x3c00", "0x3c3f", "mismatch", 43, 63, 63, "u = 63 goes to the last bin")

    aggregates = [
        {"dtype": "f32", "g": [1.0, 2.0, 3.0, 0.0], "c": [1.5, 2.0, 2.0, 0.0], "rtol": 0.4, "atol": 0.0,
         "counts": [2, 1, 1, 0, 0], "n_finite": 4, "max_abs": 1.0, "argmax_abs": 2, "max_rel": 0.5,
         "argmax_rel": 0, "max_ulp": 4194304, "argmax_ulp": 0, "sum_signed": -0.5, "sum_abs": 1.5,
         "sum_sq": 1.25, "relhist": {"0": 2, "46": 1, "47": 1}, "ulphist": {"0": 2, "63": 2},
         "mean_abs": 0.375, "var_abs": 0.171875,
         "why": "d = (0.5, 0, -1, 0); 1 <= RN32(0.4)*3; 1->1.5 and 3->2 are both 2^22 key steps (tie -> index 0); "
                "mean |d| = 1.5/4, var = 1.25/4 - (3/8)^2 = 11/64"},
        {"dtype": "f32", "g": [0.0, 0.0, 0.0], "c": [1.0, -1.0, 1.0], "rtol": 0.0, "atol": 0.0,
         "counts": [0, 0, 3, 0, 0], "n_finite": 3, "max_abs": 1.0, "argmax_abs": 0, "max_rel": float("inf"),
         "argmax_rel": 0, "max_ulp": 1065353216, "argmax_ulp": 0, "sum_signed": 1.0, "sum_abs": 3.0,
         "sum_sq": 3.0, "relhist": {"63": 3}, "ulphist": {"63": 3}, "mean_abs": 1.0, "var_abs": 0.0,
         "why": "ties resolve to the lowest index; g = 0 gives rel = +inf; |d| all 1: mean 1, variance 0"},
        {"dtype": "f16", "g": [1.0, 1.0], "c": [1.0, 1.0], "rtol": 0.0, "atol": 0.0,
         "counts": [2, 0, 0, 0, 0], "n_finite": 2, "max_abs": 0.0, "argmax_abs": 0, "max_rel": 0.0,
         "argmax_rel": 0, "max_ulp": 0, "argmax_ulp": 0, "sum_signed": 0.0, "sum_abs": 0.0, "sum_sq": 0.0,
         "relhist": {"0": 2}, "ulphist": {"0": 2}, "mean_abs": 0.0, "var_abs": 0.0,
         "why": "identical tensors: every maximum is 0 at the first finite pair"},
    ]
    out = Path(__file__).with_name("hand_cases.json")
    json.dump({"source": SEC, "cases": cases, "aggregates": aggregates}, open(out, "w"), indent=1)


if __name__ == "__main__":
    main()
