/*
 * peat_oracle.h -- TEST INFRASTRUCTURE ONLY (the oracle).
 *
 * Plain, sequential, exact CPU implementation of the PEAT error signature:
 * the element-wise error between a golden and a faulty (candidate) tensor
 * (Alg. 1 / Alg. 2 "Err(...)"; Section IV-B-3, "FI Assessment Scores":
 * the error is the absolute difference, scored by its maximum, its mean and
 * its variance) extended with the per-element relative error, the
 * ordered-integer ULP distance, a five-way classification and two 64-bin
 * histograms.  Only tests/, __graft_entry__.smoke() and bench.py's
 * cpu_baseline leg may load this code.  It shares no code with the CUDA
 * path; every declaration here is its own.
 *
 * The pseudo-error injector (Section IV-A error models: FP16 cast, random
 * value RV, random zero RZ; Section II-B: random bit flip, random NaN) is
 * restated here as well, so the device injector can be checked against it.
 */
#ifndef PEAT_ORACLE_H
#define PEAT_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* element types (codes agree with the library's dtype codes) */
enum { ORC_F32 = 0, ORC_F16 = 1, ORC_BF16 = 2, ORC_F8E4M3 = 3, ORC_F8E5M2 = 4, ORC_F64 = 5 };

/* classes, in the order of the library's class counters */
enum { ORC_EXACT = 0, ORC_WITHIN_TOL = 1, ORC_MISMATCH = 2, ORC_NAN_INF_ASYM = 3,
       ORC_SIGN_FLIP = 4, ORC_NCLASS = 5 };

/* return codes */
enum { ORC_OK = 0, ORC_BAD_ARG = 1 };

/* Per-tensor (or per-segment) signature.  Field order and types are those of
 * the first 144 bytes of the library's result record; the record's last two
 * fields (the mean and variance of |d|) are formed from the exact sums that
 * orc_compare_segmented_sums returns. */
typedef struct {
  uint64_t n;                 /* pairs compared */
  uint64_t count[ORC_NCLASS]; /* class counts */
  uint64_t n_finite;          /* pairs with both operands finite */
  double max_abs;             /* RN64 of the largest |c-g| over finite pairs */
  int64_t argmax_abs;         /* lowest index attaining it, -1 if none */
  double max_rel;             /* RN64 of the largest |c-g|/|g| (may be +inf) */
  int64_t argmax_rel;
  uint64_t max_ulp;           /* largest ULP distance over pairs without NaN */
  int64_t argmax_ulp;
  double sum_abs;             /* RN64 of the exact sum of |c-g| over finite pairs */
  double sum_sq;              /* RN64 of the exact sum of (c-g)^2 */
  double sum_signed;          /* RN64 of the exact sum of (c-g) */
  double rtol_eff, atol_eff;  /* tolerances actually used: RN32 of the inputs */
} orc_stats;

/* One tensor: g, c point to n elements of the given type.  hist receives
 * 128 counters: [0..63] log2-relative-error bins, [64..127] ULP bins. */
int orc_compare(const void* g, const void* c, int64_t n, int dtype, double rtol, double atol,
                orc_stats* st, uint64_t* hist);

/* A packed list of tensors: segment s is [offsets[s], offsets[s+1]).
 * Argmax indices are local to the segment. */
int orc_compare_segmented(const void* g, const void* c, const int64_t* offsets, int64_t nseg,
                          int dtype, double rtol, double atol, orc_stats* st, uint64_t* hist);

/* orc_compare_segmented, plus (words != NULL) the exact sums of |c-g| and of
 * (c-g)^2 over each segment's finite pairs, in the fixed-point format below:
 * segment s gets words[2 s ORC_ACC_WORDS ...] (sum |d|) followed by
 * ORC_ACC_WORDS words of sum d^2.  The Mean and Variance of Errors scores
 * (Section IV-B-3) are formed from them exactly (oracle/__init__.py). */
int orc_compare_segmented_sums(const void* g, const void* c, const int64_t* offsets, int64_t nseg,
                               int dtype, double rtol, double atol, orc_stats* st, uint64_t* hist,
                               uint64_t* words);

/* Mean of the top errors (Section IV-B-3, "Mean of Top 10% Errors"): over
 * the pairs with both operands finite, the k = ceil(n_finite * num / den)
 * largest |c - g| (0 < num <= den; the paper's score is num/den = 1/10).
 * Ties do not change the value.  All quantities exact, then RN64. */
typedef struct {
  uint64_t n_finite;  /* pairs with both operands finite */
  uint64_t k;         /* pairs taken */
  double threshold;   /* RN64 of the k-th largest |c - g| (0 if k = 0) */
  double sum;         /* RN64 of the exact sum of the k largest |c - g| */
  double mean;        /* RN64 of that exact sum divided by k (0 if k = 0) */
} orc_topk;

int orc_topk_mean(const void* g, const void* c, int64_t n, int dtype, uint64_t num, uint64_t den, orc_topk* out);

/* Context statistics of one tensor (Section IV-C-2: the means and variances
 * of the weight and activation tensors the error scores are correlated
 * with): counts, the finite minimum and maximum, and the exact sum and sum
 * of squares of the finite elements as fixed-point words (two's complement,
 * ORC_ACC_WORDS little-endian 64-bit words, least significant bit
 * 2^ORC_ACC_LSB), from which the caller forms the mean and the variance
 * exactly. */
#define ORC_ACC_WORDS 72
#define ORC_ACC_LSB (-2304)
typedef struct {
  uint64_t n, n_finite, n_nan, n_inf;
  double min, max;  /* finite extremes (0 if none) */
  uint64_t sum_words[ORC_ACC_WORDS];
  uint64_t sum_sq_words[ORC_ACC_WORDS];
} orc_tstats;

int orc_tensor_stats(const void* x, int64_t n, int dtype, orc_tstats* out);

/* ULP key of one raw bit pattern: +magnitude bits, negated when the sign
 * bit is set (so both zeros map to 0).  Exposed for the tests. */
int64_t orc_ulp_key(uint64_t bits, int dtype);

/* RN-even double of an exact rational sum of doubles, exposed so the tests
 * can check the exact accumulator against Python's exact integers:
 * returns RN64(sum_{i} x[i]) and RN64(sum_i x[i]*y[i]). */
double orc_exact_sum(const double* x, int64_t n);
double orc_exact_dot(const double* x, const double* y, int64_t n);

/* ---- pseudo-error injector ------------------------------------------- */
enum {
  ORC_INJ_RZ = 0,          /* k distinct positions set to +0 (random zero) */
  ORC_INJ_RV = 1,          /* k distinct positions get the value of a uniformly drawn element */
  ORC_INJ_BITFLIP = 2,     /* k distinct positions, one bit in [bit_lo, bit_hi] flipped */
  ORC_INJ_NAN_INF = 3,     /* Bernoulli(rate): NaN (1/2), +Inf (1/4), -Inf (1/4) */
  ORC_INJ_SIGNFLIP = 4,    /* Bernoulli(rate): sign bit flipped */
  ORC_INJ_REL_GAUSS = 5,   /* x <- RN(x * RN32(1 + sigma*z)), z ~ N(0,1) */
  ORC_INJ_ADD_GAUSS = 6,   /* x <- RN(x + sigma*z) */
  ORC_INJ_BIAS = 7,        /* x <- RN(x + alpha*|x|) */
  ORC_INJ_CAST_F16_RNE = 8, ORC_INJ_CAST_F16_RTZ = 9,   /* fp32 only: round to fp16 and back */
  ORC_INJ_CAST_BF16_RNE = 10, ORC_INJ_CAST_BF16_RTZ = 11,
  ORC_INJ_NKIND = 12
};

typedef struct {
  int32_t kind;
  int32_t k;        /* count for RZ/RV/BITFLIP */
  int32_t bit_lo;   /* BITFLIP bit range, inclusive */
  int32_t bit_hi;
  double x;         /* rate (NAN_INF, SIGNFLIP), sigma (gauss), alpha (BIAS) */
} orc_inject_model;

int orc_inject(void* dst, const void* src, int64_t n, int dtype, const orc_inject_model* models,
               int nmodels, uint64_t seed, uint64_t* counts);

/* Building blocks exposed for their own pins. */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
void orc_normal_pair_from_words(uint32_t w0, uint32_t w1, float z[2]);
float orc_logf(float x);
float orc_cos2pi(float u);
float orc_sin2pi(float u);

#ifdef __cplusplus
}
#endif
#endif
