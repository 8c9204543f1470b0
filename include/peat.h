/*
 * peat.h -- C ABI of libpeat, the GB300 (sm_103a) golden-vs-candidate error
 * signature library.
 *
 * PEAT's Analyzer scores the error between a golden tensor and a
 * fault-injected (candidate) tensor recorded during training: the error is
 * their absolute difference, scored per recorded tensor by its maximum, its
 * mean and its variance (Section IV-B-3, "FI Assessment Scores"; the Err(...)
 * step that ends Alg. 1 and Alg. 2).  This library computes that signature,
 * extended per element with the relative error, the ordered-integer ULP
 * distance and a five-way classification, in one pass over both tensors.
 *
 * Definitions (exact over the reals, then rounded once to nearest-even):
 *   non-finite pairs  EXACT if both NaN or both infinite with equal sign,
 *                     NAN_INF_ASYM otherwise; excluded from sums and from
 *                     the abs/rel maxima.
 *   finite pairs      d = c - g, a = |d|.  EXACT iff a = 0.  WITHIN_TOL iff
 *                     0 < a <= atol + rtol*|g| (torch.isclose form, golden as
 *                     reference, Section III-A; rtol/atol rounded to float32).
 *                     SIGN_FLIP iff not yet classified, g != 0, c != 0 and
 *                     the sign bits differ.  MISMATCH otherwise.
 *   relative error    a/|g|; 0 when a = 0; +inf when g = 0 < a.
 *   rel histogram     bin 0: a = 0 (and equal non-finite pairs); bins 1..62:
 *                     k = floor(log2(a/|g|)) at clamp(k+48, 1, 62); bin 63:
 *                     g = 0 < a, and every NAN_INF_ASYM pair.
 *   ULP distance      u = |key(c) - key(g)|, key(x) = +/-(bits without sign)
 *                     by the sign bit (both zeros -> 0).  Bin min(u, 63).  A
 *                     pair with a NaN has no u: bin 63 (bin 0 if both NaN),
 *                     and it is left out of max_ulp.
 *   maxima            lowest index wins ties (exact comparison).
 *   sums              over finite pairs: sum |d|, sum d^2, sum d, exact, then
 *                     rounded to nearest-even binary64.
 * Derived scores (host side): mean = sum_abs/n_finite, bias =
 * sum_signed/n_finite, L2 = sqrt(sum_sq), variance of |e| =
 * sum_sq/n_finite - mean^2.
 *
 * Conventions for every entry point
 *  - Pointers named golden/candidate/src/dst/stats_out/hist_out/counts_out
 *    are DEVICE pointers (cudaMalloc or managed memory) owned by the caller;
 *    `offsets` and `models` are HOST arrays the call copies before returning.
 *  - Every call is asynchronous on `stream` (NULL = legacy default stream);
 *    outputs are valid once the stream has been synchronised.
 *  - A handle is not thread-safe: use one handle per host thread.  Calls on
 *    one handle must not overlap on the GPU (the handle's workspace is reused
 *    call after call; issue them on one stream, or order the streams).
 *  - Errors are returned as peat_status_t; nothing is thrown across the ABI.
 *    peat_last_error(h) gives the text of the last error on that handle.
 *    CUDA errors map to PEAT_ERR_CUDA.
 */
#ifndef PEAT_H
#define PEAT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A CUDA stream (layout-compatible with cudaStream_t / CUstream). */
typedef struct CUstream_st* peat_stream_t;

/* Element types.  The 8-bit ones are the OCP FP8 formats: E4M3 ("fn": exponent
 * bias 7, no infinities, S.1111.111 the only NaN, 448 the largest value) and
 * E5M2 (bias 15, IEEE-like infinities and NaNs); peat_compare,
 * peat_compare_segmented and peat_isclose_grid take them.  PEAT_F64
 * (IEEE binary64, e.g. a float32 output widened exactly to compare with a
 * binary64 one) is taken by the same three; its ULP distance counts binary64
 * steps and its sums may round to +-inf.  The other entry points return
 * PEAT_ERR_UNSUPPORTED for these types. */
typedef enum {
  PEAT_F32 = 0,
  PEAT_F16 = 1,
  PEAT_BF16 = 2,
  PEAT_F8E4M3 = 3,
  PEAT_F8E5M2 = 4,
  PEAT_F64 = 5
} peat_dtype_t;

typedef enum {
  PEAT_OK = 0,
  PEAT_ERR_INVALID_ARG = 1, /* null pointer, negative size, bad dtype, bad offsets, ... */
  PEAT_ERR_UNSUPPORTED = 2, /* a valid request the library does not serve */
  PEAT_ERR_ALLOC = 3,       /* device or pinned allocation failed */
  PEAT_ERR_CUDA = 4,        /* a CUDA runtime call failed (text in peat_last_error) */
  PEAT_ERR_TIMEOUT = 5,     /* a bounded device-side wait expired */
  PEAT_ERR_INTERNAL = 6     /* an internal consistency check failed: an exact
                               accumulator of an earlier call needed a digit
                               outside its range (the kernels never write it out
                               of bounds but raise a library-wide mapped status
                               word; the next handle call of any handle, or the
                               next peat_compare_noalloc, returns this once and
                               clears it; the outputs since the previous check
                               are invalid) */
} peat_status_t;

/* Classes, in the order of peat_stats_t.count. */
enum {
  PEAT_EXACT = 0,
  PEAT_WITHIN_TOL = 1,
  PEAT_MISMATCH = 2,
  PEAT_NAN_INF_ASYM = 3,
  PEAT_SIGN_FLIP = 4,
  PEAT_NCLASS = 5
};

/* Tolerances of the WITHIN_TOL test; both are rounded to float32 (round to
 * nearest even) and must then be finite and >= 0. */
typedef struct {
  double rtol;
  double atol;
} peat_tol_t;

/* Handle configuration.  device: CUDA ordinal the handle's calls run on.
 * max_segments: the largest nseg a segmented call may pass (0 = 4096).
 * flags: 0, or PEAT_FLAG_TEST_EXPIRE_WAITS. */
typedef struct {
  int32_t device;
  int32_t reserved0;
  int64_t max_segments;
  uint32_t flags;
  uint32_t reserved1;
} peat_config_t;

/* Testing aid: every bounded device-side wait of the compare pipeline gives
 * up at its first poll, so the timeout path (error flag, drained copies,
 * PEAT_ERR_TIMEOUT on the next call) can be exercised without a real stall.
 * Outputs of calls on such a handle are not valid. */
#define PEAT_FLAG_TEST_EXPIRE_WAITS 0x80000000u

/* Signature of one tensor (or one segment).  160 bytes, no padding holes. */
typedef struct {
  uint64_t n;                   /* pairs compared */
  uint64_t count[PEAT_NCLASS];  /* class counts; they sum to n */
  uint64_t n_finite;            /* pairs with both operands finite */
  double max_abs;               /* RN64(max |d|) over finite pairs, 0 if none */
  int64_t argmax_abs;           /* lowest index attaining it, -1 if no finite pair */
  double max_rel;               /* RN64(max a/|g|) over finite pairs; may be +inf */
  int64_t argmax_rel;           /* -1 if no finite pair */
  uint64_t max_ulp;             /* max u over pairs without a NaN */
  int64_t argmax_ulp;           /* -1 if every pair has a NaN */
  double sum_abs;               /* RN64(sum |d|) over finite pairs */
  double sum_sq;                /* RN64(sum d^2) */
  double sum_signed;            /* RN64(sum d) */
  double rtol_eff;              /* the float32 tolerances actually used */
  double atol_eff;
  /* The paper's Mean and Variance of Errors scores (Section IV-B-3) over the
   * n_finite pairs, each the exact value rounded once (RN-even binary64,
   * computed on the device from the exact sums; 0 if n_finite = 0):
   *   mean_abs = sum |d| / n_finite,
   *   var_abs  = (n_finite sum d^2 - (sum |d|)^2) / n_finite^2 (population). */
  double mean_abs;
  double var_abs;
} peat_stats_t;

/* Histograms of one tensor: 128 uint64 counters, [0..63] log2-relative-error
 * bins then [64..127] ULP bins.  Each half sums to n. */
#define PEAT_HIST_BINS 128

typedef struct peat_handle_s* peat_handle_t;

/* Create a handle bound to cfg->device (cfg may be NULL: device 0, defaults).
 * Allocates the handle's device workspace.  Errors: INVALID_ARG, CUDA, ALLOC. */
peat_status_t peat_signature_create(peat_handle_t* out, const peat_config_t* cfg);

/* Release the handle and its workspace; waits for the handle's work to finish.
 * NULL is accepted and ignored. */
peat_status_t peat_signature_destroy(peat_handle_t h);

/* Signature of one tensor pair (the Err step of Alg. 1 / Alg. 2 over one
 * recorded tensor; scores of Section IV-B-3).
 *   golden, candidate  device arrays of n elements of `dtype`, any alignment
 *                      (16-byte aligned arrays with equal alignment run the
 *                      vectorised path); contiguous, element i at byte
 *                      i*sizeof(dtype).
 *   n                  >= 0; n = 0 yields zero counts and argmax -1.
 *   tol                see peat_tol_t.
 *   stats_out          device pointer to one peat_stats_t.
 *   hist_out           device pointer to PEAT_HIST_BINS uint64 (or NULL).
 * Errors: INVALID_ARG (null pointer with n > 0, n < 0, bad dtype, bad tol),
 * CUDA, TIMEOUT (a bounded device wait of an EARLIER call on this handle
 * expired; that call's outputs are invalid; the flag is cleared). */
peat_status_t peat_compare(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                           peat_dtype_t dtype, peat_tol_t tol, peat_stats_t* stats_out,
                           uint64_t* hist_out, peat_stream_t stream);

/* Per-segment signatures of a packed list of tensors (e.g. every parameter
 * of a model, recorded per epoch as in Alg. 1).  Segment s is elements
 * [offsets[s], offsets[s+1]) of golden/candidate; argmax indices are local
 * to the segment.
 *   offsets    HOST array of nseg+1 int64, offsets[0] = 0, non-decreasing;
 *              copied during the call.  Empty segments are allowed.
 *   nseg       0 <= nseg <= the handle's max_segments.
 *   stats_out  device array of nseg peat_stats_t.
 *   hist_out   device array of nseg*PEAT_HIST_BINS uint64 (or NULL).
 * Errors: INVALID_ARG (as above, or offsets not non-decreasing from 0),
 * UNSUPPORTED (nseg above max_segments), CUDA. */
peat_status_t peat_compare_segmented(peat_handle_t h, const void* golden, const void* candidate,
                                     const int64_t* offsets, int64_t nseg, peat_dtype_t dtype,
                                     peat_tol_t tol, peat_stats_t* stats_out, uint64_t* hist_out,
                                     peat_stream_t stream);

/* Pseudo-error models (Section IV-A: FP16 cast, random value RV, random zero
 * RZ with num_pos positions; Section II-B: random bit flip, random NaN; plus
 * multiplicative and additive Gaussian noise, a relative bias and sign flips). */
typedef enum {
  PEAT_INJ_RZ = 0,        /* k distinct positions set to +0 */
  PEAT_INJ_RV = 1,        /* k distinct positions take the value of a uniformly drawn element of src */
  PEAT_INJ_BITFLIP = 2,   /* k distinct positions, one bit in [bit_lo, bit_hi] flipped */
  PEAT_INJ_NAN_INF = 3,   /* each element with probability x: NaN (1/2), +Inf (1/4), -Inf (1/4) */
  PEAT_INJ_SIGNFLIP = 4,  /* each element with probability x: sign bit flipped */
  PEAT_INJ_REL_GAUSS = 5, /* v <- RN(v * RN32(1 + x*z)), z ~ N(0,1) */
  PEAT_INJ_ADD_GAUSS = 6, /* v <- RN(RN32(v + x*z)) */
  PEAT_INJ_BIAS = 7,      /* v <- RN(RN32(v + x*|v|)) */
  PEAT_INJ_CAST_F16_RNE = 8, /* float32 tensors only: round to binary16 (nearest even) and back */
  PEAT_INJ_CAST_F16_RTZ = 9, /* ... toward zero */
  PEAT_INJ_CAST_BF16_RNE = 10,
  PEAT_INJ_CAST_BF16_RTZ = 11
} peat_inject_kind_t;

typedef struct {
  int32_t kind;   /* peat_inject_kind_t */
  int32_t k;      /* RZ/RV/BITFLIP: number of distinct positions, 0 <= k <= min(n, 2^20) */
  int32_t bit_lo; /* BITFLIP: inclusive bit range within the element */
  int32_t bit_hi;
  double x;       /* NAN_INF/SIGNFLIP: probability in [0,1]; GAUSS: sigma; BIAS: alpha (rounded to float32) */
} peat_inject_t;

/* Seeded pseudo-error generator (the Inject step of Alg. 1 / Alg. 2).
 * dst = src with models[0..nmodels) applied in array order; each model sees
 * the previous model's output, except that RV copies from src.  Noise,
 * bias and cast models leave NaN/Inf elements unchanged.  Randomness is
 * Philox4x32-10 keyed by `seed`: element i of model m uses counter
 * (i lo, i hi, m, 0x454C454D); the j-th position draw of a fixed-count model
 * uses (j lo, j hi, m, 0x504F5331).  Results are bit-identical run to run.
 *   dst, src     device arrays of n elements (dst == src allowed; partial
 *                overlap is not).
 *   models       HOST array of nmodels (0 <= nmodels <= 64).
 *   counts_out   device array of nmodels uint64: how many elements each
 *                model fired on (k for the fixed-count models; the number
 *                of finite elements for noise/bias/cast).
 * Errors: INVALID_ARG (bad model parameters, cast on a non-float32 tensor,
 * k > n), CUDA, ALLOC. */
peat_status_t peat_pseudo_error_inject(peat_handle_t h, void* dst, const void* src, int64_t n,
                                       peat_dtype_t dtype, const peat_inject_t* models, int nmodels,
                                       uint64_t seed, uint64_t* counts_out, peat_stream_t stream);

/* Fused pseudo-error assessment of one tensor (the Inject and Compare steps
 * of the playback loop, Alg. 1, in one read of the golden tensor): the
 * candidate is golden with models[0..nmodels) applied in array order, each
 * element generated in registers and never written to memory, and the result
 * is that of peat_compare(golden, candidate) with the candidate
 * peat_pseudo_error_inject(golden, models, seed) would write, bit for bit.
 *   golden        device array of n elements (any alignment).
 *   models        HOST array, 1 <= nmodels <= 8, element-wise kinds only
 *                 (NAN_INF, SIGNFLIP, REL_GAUSS, ADD_GAUSS, BIAS, the casts);
 *                 parameters as for peat_pseudo_error_inject.
 *   seed          the injector's seed (same Philox counters).
 *   tol, stats_out, hist_out  as for peat_compare.
 * No per-model fire counts are produced.
 * Errors: INVALID_ARG (as for the two calls it fuses), UNSUPPORTED (a
 * fixed-count model: RZ, RV, BITFLIP draw their positions on the host and
 * are applied by peat_pseudo_error_inject), CUDA, ALLOC. */
peat_status_t peat_inject_compare(peat_handle_t h, const void* golden, int64_t n, peat_dtype_t dtype,
                                  const peat_inject_t* models, int nmodels, uint64_t seed, peat_tol_t tol,
                                  peat_stats_t* stats_out, uint64_t* hist_out, peat_stream_t stream);

/* Mean of the top errors of one tensor pair (Section IV-B-3, "Mean of Top
 * 10% Errors").  48 bytes. */
typedef struct {
  uint64_t n_finite;  /* pairs with both operands finite */
  uint64_t k;         /* pairs taken: ceil(n_finite * num / den) */
  double threshold;   /* RN64 of the k-th largest |c - g| (0 if k = 0) */
  double sum;         /* RN64 of the exact sum of the k largest |c - g| */
  double mean;        /* RN64 of that exact sum divided by k (0 if k = 0) */
  uint32_t exact;     /* always 1: every field is exact as defined (kept for the layout) */
  uint32_t reserved;
} peat_topk_t;

/* Mean of the top errors: over the pairs with both operands finite, the
 * k = ceil(n_finite * num / den) largest |c - g| (0 < num <= den; the paper's
 * score is num/den = 1/10), their exact sum and its exact mean, each rounded
 * once to nearest-even binary64.  Ties do not change the value.
 *   golden, candidate  as for peat_compare (device, any alignment).
 *   out                device pointer to one peat_topk_t.
 * Streams both tensors three times (a radix select over an order-preserving
 * key of |c - g|, 10 + 11 + 10 bits, that sums exactly what it has resolved
 * as it goes), a fourth time only when more than 65536 pairs whose |c - g| is
 * not a float32 value lie within 1024 float32 steps of the k-th largest, and
 * a fifth and sixth time only when more than 65536 of them share the float32
 * rounding of the k-th largest (a radix select over their rounding errors);
 * asynchronously on `stream`.  The handle's workspace is shared with its
 * other calls (do not overlap them).
 * Errors: INVALID_ARG (null pointer with n > 0, n < 0, bad dtype, num = 0,
 * num > den, out NULL), UNSUPPORTED (more than 2^24 elements per thread of the
 * grid: n above about 2^42 on a 152-SM GPU), CUDA. */
peat_status_t peat_topk_mean(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                             peat_dtype_t dtype, uint64_t num, uint64_t den, peat_topk_t* out,
                             peat_stream_t stream);

/* torch.isclose pass counts over a grid of tolerances (Section III-A; its
 * Fig. 5 plots the share of output elements isclose accepts for FP16-FP32
 * and FP32-FP64 pairs as rtol and atol vary), in one read of both tensors:
 * counts_out[i * na + j] = the pairs peat_compare with tolerance
 * (rtols[i], atols[j]) would class EXACT or WITHIN_TOL, i.e. both operands
 * NaN, or the same infinity, or finite with |c - g| <= atols[j] + rtols[i] |g|
 * exactly.
 *   golden, candidate  as for peat_compare (device, any alignment).
 *   rtols, atols       HOST arrays (read before return); every value finite
 *                      and >= 0, rounded to float32 as peat_compare does;
 *                      rtols non-decreasing after the rounding.
 *   nr, na             1 <= nr, na and nr * na <= 64.
 *   counts_out         device pointer to nr * na uint64 (overwritten).
 * About 15 na log2(nr) operations per differing pair (a binary search per
 * atol, bounded by the previous atol's result; bitwise-equal warp slots cost
 * a vote).  Asynchronous on `stream`.
 * Errors: INVALID_ARG (bad dtype, pointers, tolerances or grid size), CUDA. */
peat_status_t peat_isclose_grid(peat_handle_t h, const void* golden, const void* candidate, int64_t n,
                                peat_dtype_t dtype, const double* rtols, int nr, const double* atols, int na,
                                uint64_t* counts_out, peat_stream_t stream);

/* Context statistics of one recorded tensor (Section IV-C-2: the means and
 * variances of the weight and activation tensors that the error scores are
 * correlated with).  80 bytes.  Every double is the exact value rounded once
 * to nearest-even. */
typedef struct {
  uint64_t n;         /* elements */
  uint64_t n_finite;  /* finite elements */
  uint64_t n_nan;     /* NaN elements */
  uint64_t n_inf;     /* infinite elements */
  double sum;         /* sum of the finite elements */
  double sum_sq;      /* sum of their squares */
  double mean;        /* sum / n_finite (0 if n_finite = 0) */
  double var;         /* population variance: (n_finite sum_sq - sum^2) / n_finite^2, exact
                         before its one rounding (0 if n_finite = 0) */
  double min, max;    /* smallest and largest finite element (0 if none) */
} peat_tstats_t;

/* Context statistics of each segment s = [offsets[s], offsets[s+1]) of x
 * (a single tensor: offsets = {0, n}, nseg = 1).
 *   x           device pointer, dtype elements, any alignment.
 *   offsets     HOST array of nseg + 1 non-decreasing int64, offsets[0] = 0;
 *               copied before return.
 *   stats_out   device pointer to nseg peat_tstats_t.
 * Streams x once (about 25 integer operations per element), then one thread
 * per segment forms the mean and the variance from the exact sums.
 * Asynchronous on `stream`; shares the handle's workspace with its other
 * calls (do not overlap them).
 * Errors: INVALID_ARG (bad dtype, offsets, null pointers), UNSUPPORTED (nseg
 * above the handle's max_segments, a segment of 2^36 elements or more), CUDA. */
peat_status_t peat_tensor_stats(peat_handle_t h, const void* x, const int64_t* offsets, int64_t nseg,
                                peat_dtype_t dtype, peat_tstats_t* stats_out, peat_stream_t stream);

/* Host-side Analyzer steps (Section IV-C).  No GPU work; x and y are HOST
 * arrays of finite doubles.
 *
 * peat_spearman: Spearman rank correlation of x and y (Section IV-C-2): the
 *   Pearson correlation of their ranks, tied values taking the mean of the
 *   ranks they span.  *rho_out = NaN when n < 2 or either ranking is constant.
 *   The rank sums are exact integers; rho is their exact ratio up to the one
 *   square root and division (a few ulps).
 * peat_mean_std: the model-wise error range of one layer (Section IV-C-1): the
 *   mean and the standard deviation of its scores across epochs, with ddof 0
 *   (population) or 1 (sample); std = NaN when n <= ddof, mean = NaN when
 *   n = 0.
 * Errors: INVALID_ARG (null pointer, n < 0, a non-finite value, ddof not 0 or
 *   1); text in peat_last_error(NULL). */
peat_status_t peat_spearman(const double* x, const double* y, int64_t n, double* rho_out);
peat_status_t peat_mean_std(const double* x, int64_t n, int ddof, double* mean_out, double* std_out);

/* The cross-step trend of an error score over replayed epochs (Alg. 1 runs
 * the Err step once per recorded epoch; Section IV-C-1 reads each layer's
 * scores across epochs): the least-squares line log y = intercept +
 * slope log x through the points (x[i], y[i]) with x[i] > 0 and y[i] > 0
 * finite (the others, e.g. a step whose score is 0, are left out), so that
 * y ~ exp(intercept) x^slope; an error growing like sqrt(step) gives slope
 * 1/2.  Two passes over the log values with compensated sums (host code).
 *   slope_out, intercept_out  NaN when fewer than two points remain or all
 *                             their x are equal;
 *   r2_out                    the fit's coefficient of determination, NaN
 *                             when all remaining log y are equal;
 *   used_out                  the number of points used (may be NULL).
 * Errors: INVALID_ARG (null pointer, n < 0); text in peat_last_error(NULL). */
peat_status_t peat_trend(const double* x, const double* y, int64_t n, double* slope_out, double* intercept_out,
                         double* r2_out, int64_t* used_out);

/* Text of the last error reported on h (never NULL; "" if none).  With
 * h == NULL, the last error on this thread of the calls that take no handle
 * (peat_signature_create, peat_compare_noalloc, peat_spearman,
 * peat_mean_std, peat_trend), whichever failed last. */
const char* peat_last_error(peat_handle_t h);

/* peat_compare without a handle and without any allocation.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate at
 * the moment they compare, for instance
 *   - code whose device memory is wholly owned by a pool or caching allocator
 *     (a framework at its memory limit, or a handler comparing tensors after
 *     an out-of-memory error), where a new cudaMalloc fails or evicts;
 *   - timing-sensitive loops, where cudaMalloc/cudaFree would synchronise the
 *     device and stall every stream;
 * and it does not need a handle (creating one allocates its workspace).
 *
 * Arguments and outputs are those of peat_compare (one tensor, no segments)
 * for PEAT_F32, PEAT_F16 and PEAT_BF16 operands; PEAT_F64, PEAT_F8E4M3 and
 * PEAT_F8E5M2 return PEAT_ERR_UNSUPPORTED.  Instead of a handle's workspace
 * it uses one fixed block of device memory per device, reserved when the
 * library's device code is loaded (about 21 MB: per-CTA lists of
 * general-path pairs for up to 320 CTAs, their partial results, the CTA
 * bounds, a status word and one accumulator).  Nothing is allocated by a
 * call, on the device or on the host.
 *   - Each CTA's range must stay below 2^31 - 64 elements (at most 320
 *     CTAs, two per SM): a larger n is rejected with PEAT_ERR_UNSUPPORTED.
 *   - The block's accumulator must be zero when a call starts.  It is zero
 *     when the code loads and every call that runs to completion leaves it
 *     zero; a call that fails to launch clears it with cudaMemsetAsync.
 *   - All calls on one device share the block: two calls that overlap on the
 *     GPU (different streams without ordering, or different host threads)
 *     race and both results are invalid.  Order them on one stream.
 *   - The first call on each device does a one-time setup (it looks up the
 *     block's address with cudaGetSymbolAddress and sets kernel attributes);
 *     make it before any stream capture.
 *   - It launches two kernels on `stream`: the CTA bounds (which also
 *     clears the block's status word), then the compare.
 *   - A bounded device-side wait that expires leaves the outputs invalid and
 *     marks them: argmax_abs, argmax_rel and argmax_ulp are then -2 (a value
 *     no valid call produces).  peat_compare marks them the same way and also
 *     reports PEAT_ERR_TIMEOUT on the handle's next call.
 * Errors: as peat_compare, plus PEAT_ERR_UNSUPPORTED (n, dtype or device
 * ordinal beyond the limits); the text is in peat_last_error(NULL). */
peat_status_t peat_compare_noalloc(const void* golden, const void* candidate, int64_t n, peat_dtype_t dtype,
                                   peat_tol_t tol, peat_stats_t* stats_out, uint64_t* hist_out,
                                   peat_stream_t stream);

/* Profiling aid: with event != NULL (a cudaEvent_t created on h's device),
 * every later peat_compare, peat_compare_segmented and peat_inject_compare
 * call on h records it on the call's stream right after enqueuing stage 1,
 * i.e. before the per-segment finalize launch of a multi-segment call (a
 * one-segment call finalizes inside stage 1).  Events recorded around the
 * call then time stage 1 alone and the finalize alone.  NULL stops it.  The
 * event must outlive its use.  Errors: INVALID_ARG (h NULL). */
peat_status_t peat_set_stage1_event(peat_handle_t h, void* event);

/* Testing aid for peat_compare_noalloc (the counterpart of
 * PEAT_FLAG_TEST_EXPIRE_WAITS): on != 0 makes every bounded device-side wait
 * of later calls give up at its first poll, so that the expired-wait marking
 * can be exercised without a real stall; on = 0 restores the normal limit. */
void peat_test_noalloc_expire_waits(int on);

/* Testing aid for the range check of the exact accumulators (runs on the
 * host, no GPU involved): the kernels' split of +-m 2^e (m = m_hi 2^64 +
 * m_lo, neg != 0 for the minus sign) into the signed 32-bit digits of their
 * fixed-point sums.  digits_out (24 entries) receives the digit of weight
 * 2^(32 j - 416) at index j.  Returns 1 if a nonzero digit fell outside those
 * 24 (it is not written; the kernels report this case as PEAT_ERR_INTERNAL),
 * else 0. */
int32_t peat_test_for_digits(uint64_t m_lo, uint64_t m_hi, int32_t e, int32_t neg, int64_t* digits_out);

/* Testing aid for the one rounding of the Mean and Variance of Errors scores
 * (runs on the host, no GPU involved): RN-even binary64 of (W + f) 2^e / d
 * with W = w_hi 2^64 + w_lo (w_hi's top bit set), 0 < f < 1 when sticky != 0
 * and f = 0 otherwise, 1 <= d < 2^64 -- the routine the kernels round both
 * scores with.  NaN for arguments outside that domain. */
double peat_test_quot_rn(uint64_t w_hi, uint64_t w_lo, int32_t sticky, int32_t e, uint64_t d);

#ifdef __cplusplus
}
#endif
#endif /* PEAT_H */
