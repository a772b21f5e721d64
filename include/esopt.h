/*
 * esopt.h -- C ABI of the GB300 (sm_103a) library for the parameter-space
 * evolution-strategies (ES) step of Agentic ESOpt.
 *
 * One ES generation as the paper states it (§3, §3.1, App. D.6):
 *
 *   sigma_t = cosine schedule (§3.1)                       es_sigma_cosine
 *   for each member i with integer seed s_i:
 *       theta <- theta + sigma_t * eps_{s_i}   (in place)   es_perturb
 *       R_i   <- rollout(theta)                (caller)
 *       theta <- theta - sigma_t * eps_{s_i}   (in place)   es_restore
 *   Rhat  <- population z-score of R (§3)                  es_normalize_rewards
 *   c_i   <- alpha * Rhat_i / G  (§3; optionally / sigma)  es_update_coeffs
 *   theta <- theta + sum_i c_i * eps_{s_i}    (one pass)    es_update
 *
 * The noise eps_s is never stored. Per member only its integer seed is kept,
 * and the noise is regenerated from it whenever it is needed (§3; App. D.6).
 * The paper does not name a generator; this library fixes it as follows, for
 * every entry point:
 *
 *   block j = floor(g / 4) of global parameter index g,
 *   Philox4x32-10 (Salmon et al., SC'11) with key = (seed_lo32, seed_hi32) and
 *   counter = (j_lo32, j_hi32, 0, 0) -> 32-bit words x0, x1, x2, x3,
 *   u(x) = (2 * (x >> 9) + 1) / 2^24, in (0, 1),
 *   eps[4j+0] = r01 cos(2 pi u(x1)),  eps[4j+1] = r01 sin(2 pi u(x1)),
 *   eps[4j+2] = r23 cos(2 pi u(x3)),  eps[4j+3] = r23 sin(2 pi u(x3)),
 *   with r01 = sqrt(-2 ln u(x0)) and r23 = sqrt(-2 ln u(x2)) (Box-Muller).
 *
 * Device values are computed in fp32 and agree with the exact definition to
 * |delta eps| <= 1e-5 * max(1, |eps|). Every device entry point derives eps
 * from bit-identical radius and angle values, and applies a scale s as
 * fma(-(s * r), cos, theta) (resp. sin), so es_restore adds exactly the
 * negation of es_perturb's increment (it undoes it up to the storage
 * rounding) and es_update uses the same directions that were evaluated.
 *
 * Conventions for every function:
 *   - All device memory (parameters, noise buffers) belongs to the caller. The
 *     library allocates only a plan's device copy of its segment table.
 *   - Device entry points are asynchronous on `stream`, a cudaStream_t passed
 *     as void* (NULL = the legacy default stream), and run on the device that is
 *     current on the calling thread. Host arrays passed to them (seeds,
 *     coefficients) may be reused as soon as the call returns.
 *   - Errors are returned as es_status_t; no exception crosses the ABI. A CUDA
 *     launch error returns ES_ERR_CUDA; es_last_error() gives the detail. An
 *     asynchronous fault of an earlier launch surfaces at the caller's next
 *     synchronisation.
 *   - Results do not depend on the launch configuration: each element's value
 *     is a function of (seed, global index, its old value, scalars) only, so
 *     repeated calls give bit-identical parameters on every run.
 *   - Thread safety: distinct plans may be used from different threads; one plan
 *     must not be used on two streams at once.
 *   - Plan-based device entry points neither synchronise the host nor allocate
 *     per call, so they can be recorded in a CUDA graph (stream capture); the
 *     host arguments of a captured call (seeds, coefficients, sigma) are fixed
 *     at capture time.
 */
#ifndef ESOPT_H_
#define ESOPT_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Largest population (number of seeds) one es_update call accepts, and the
   largest number of seeds one generation of es_replay may have. */
#define ES_MAX_SEEDS 1024

typedef enum {
  ES_OK = 0,
  ES_ERR_INVALID_ARG = 1,    /* null pointer, n < 1, bad enum, empty segment   */
  ES_ERR_ALIGNMENT = 2,      /* segment data not 16-byte aligned, index base
                                not a multiple of 8, noise buffer not 4-byte
                                aligned                                       */
  ES_ERR_OVERLAP = 3,        /* two segments share memory or index ranges     */
  ES_ERR_NONFINITE = 4,      /* sigma or a coefficient is NaN or infinite     */
  ES_ERR_TOO_MANY_SEEDS = 5, /* n > ES_MAX_SEEDS                              */
  ES_ERR_CUDA = 6,           /* a CUDA runtime call or kernel launch failed   */
  ES_ERR_NO_MEMORY = 7,      /* host or device allocation failed              */
  ES_ERR_WRONG_DEVICE = 8    /* plan used while another device is current     */
} es_status_t;

/*
 * Storage type of the parameters. Arithmetic is fp32 in every case.
 * ES_FP8_E4M3 stores each element as an 8-bit E4M3 float (OCP 8-bit floating
 * point: 4 exponent bits with bias 7, 3 mantissa bits, subnormals, no
 * infinities, largest finite value 448) times a scale per segment
 * (es_plan_create_scaled); results are rounded to the nearest E4M3 value,
 * ties to even, saturating at +-448. The paper leaves ES on quantized weights
 * as future work (App. A.2); this storage type changes only the grid the
 * parameters are rounded to, not the step.
 */
typedef enum { ES_BF16 = 0, ES_FP32 = 1, ES_FP8_E4M3 = 2 } es_dtype_t;

/* Scale of the update coefficients (es_update_coeffs). */
typedef enum {
  /* c_i = alpha * Rhat_i / G: the implemented update of §3 (restated in
     App. D.6), which omits 1/sigma and lets alpha set the step size. */
  ES_SCALE_PAPER = 0,
  /* c_i = alpha * Rhat_i / (G * sigma): the canonical Monte Carlo estimator of
     the ES gradient, Eq. (4) and App. C.1. */
  ES_SCALE_CANONICAL = 1
} es_scale_t;

/*
 * One parameter tensor of the full parameter set (the perturbation reaches
 * every tensor of the model, §3 and App. D.6).
 *   data        device pointer to `numel` contiguous elements of the plan's
 *               dtype; must be 16-byte aligned; owned by the caller and must
 *               stay valid while the plan is used.
 *   numel       number of elements, >= 1.
 *   index_base  global parameter index of data[0]; element k has global index
 *               index_base + k, which keys its noise. Must be a multiple of 8.
 *               Index ranges of a plan's segments must not overlap.
 */
typedef struct {
  void* data;
  uint64_t numel;
  uint64_t index_base;
} es_segment_t;

typedef struct es_plan* es_plan_t;

/*
 * Validates the segment list and copies it to the current device (one
 * cudaMalloc of about 32 bytes per segment; synchronous). Every segment must
 * lie in device (or managed) memory of the current device: host pointers,
 * page-locked or not, are rejected with ES_ERR_INVALID_ARG, since a kernel
 * given one could fault. The segment list itself may
 * be freed after the call. The plan is immutable.
 * Errors: ES_ERR_INVALID_ARG (segs or out NULL, nseg < 1, numel 0, bad dtype,
 * index range past 2^64), ES_ERR_ALIGNMENT, ES_ERR_OVERLAP,
 * ES_ERR_NO_MEMORY, ES_ERR_CUDA. On error *out is set to NULL.
 */
es_status_t es_plan_create(const es_segment_t* segs, int nseg, es_dtype_t dtype,
                           es_plan_t* out);

/*
 * A plan whose segments carry one scale each: element k of segment j has the
 * value scales[j] * stored[k]. For ES_FP8_E4M3 storage, whose range and
 * spacing are fixed, the scale places a tensor's values on the E4M3 grid (a
 * per-tensor scale such as max|w| / 448). Every device entry point then works
 * on the scaled values: a perturb adds sigma * eps to scales[j] * stored[k]
 * and stores the nearest E4M3 value of the result divided by scales[j].
 * scales is a host array of nseg finite values > 0 whose reciprocals are
 * finite; it may be freed after the call. es_plan_create on ES_FP8_E4M3
 * segments uses scale 1 for every segment. Only ES_FP8_E4M3 takes scales.
 * Segment rules and errors as es_plan_create, and ES_ERR_INVALID_ARG for a
 * NULL, non-finite or non-positive scale or another dtype.
 */
es_status_t es_plan_create_scaled(const es_segment_t* segs, const float* scales, int nseg,
                                  es_dtype_t dtype, es_plan_t* out);

/* Frees the plan's device table (synchronises the device). NULL is a no-op. */
es_status_t es_plan_destroy(es_plan_t plan);

/* Total number of parameters in the plan (0 for NULL). */
uint64_t es_plan_numel(es_plan_t plan);

/*
 * Assigns index_base to each segment in order: the first gets 0, each next one
 * the previous base + numel rounded up to a multiple of 8. Returns the end of
 * the index range (the last base + numel), or 0 if the range would pass 2^64
 * (then the bases are only partly assigned). Host-only, pure.
 */
uint64_t es_assign_index_bases(es_segment_t* segs, int nseg);

/*
 * out[k] = eps_seed[index_base + k] for k in [0, n), as fp32 on the device.
 * Any index_base and n (n = 0 is a no-op); `out` must be device memory of the
 * current device, 4-byte aligned, and index_base + n must not pass 2^64.
 * Regenerates exactly the values the other device entry points use: the update
 * rebuilds each member's direction from its seed alone (App. D.6).
 */
es_status_t es_noise_fill(uint64_t seed, uint64_t index_base, uint64_t n,
                          float* out, void* stream);

/*
 * Raw generator words behind every device entry point:
 * out[4t + w] = word w (0..3) of Philox4x32-10 block (block_base + t) of
 * `seed`, for t in [0, nblocks); block j holds the noise of global indices
 * 4j .. 4j+3. For checking the integer stream bit for bit (reproducibility
 * across runs, devices and implementations). `out` is a buffer of
 * 4 * nblocks words in device memory of the current device and must be
 * 16-byte aligned; nblocks = 0 is a no-op and block_base + nblocks must not
 * pass 2^62.
 * Errors: ES_ERR_INVALID_ARG, ES_ERR_ALIGNMENT, ES_ERR_CUDA.
 */
es_status_t es_noise_bits(uint64_t seed, uint64_t block_base, uint64_t nblocks,
                          uint32_t* out, void* stream);

/*
 * The uniform mapping and Box-Muller transform of the generator applied to
 * caller-supplied word pairs, in fp32, exactly as every device entry point
 * applies them to Philox words:
 *   out[2k]   = r cos(2 pi u(words[2k+1])),  out[2k+1] = r sin(2 pi u(words[2k+1])),
 *   r = sqrt(-2 ln u(words[2k])),  u(x) = (2 (x >> 9) + 1) / 2^24.
 * Each word matters only through its top 23 bits, so this lets the transform
 * be checked over its whole input domain. `words` and `out` are buffers of
 * 2 * npairs entries in device memory of the current device, 8-byte aligned;
 * npairs = 0 is a no-op.
 * Errors: ES_ERR_INVALID_ARG, ES_ERR_ALIGNMENT, ES_ERR_CUDA.
 */
es_status_t es_box_muller(const uint32_t* words, uint64_t npairs, float* out, void* stream);

/*
 * Perturb in place, theta + sigma_t eps_i before member i's rollout (§3;
 * App. D.6):
 * theta[g] <- round(theta[g] + sigma * eps_seed[g]) for every element of every
 * segment, with the product and sum in fp32 (one fused multiply-add) and one
 * rounding to the storage type (round to nearest even).
 * Errors: ES_ERR_INVALID_ARG (NULL plan), ES_ERR_NONFINITE (sigma),
 * ES_ERR_WRONG_DEVICE, ES_ERR_CUDA.
 */
es_status_t es_perturb(es_plan_t plan, uint64_t seed, float sigma, void* stream);

/*
 * Restore in place after the rollout: the perturbation is subtracted from the
 * same buffer it was added to (§3; App. D.6):
 * theta[g] <- round(theta[g] - sigma * eps_seed[g]), same seed and sigma as the
 * es_perturb it undoes. In fp32 storage the round trip returns theta to within
 * one rounding; in bf16 an element can end one ulp away where theta + sigma*eps
 * crossed a power of two. Errors as es_perturb.
 */
es_status_t es_restore(es_plan_t plan, uint64_t seed, float sigma, void* stream);

/*
 * Restore one member and perturb the next in a single pass over theta:
 *   theta[g] <- round(round(theta[g] - sigma_restore * eps_{restore_seed}[g])
 *                     + sigma_perturb * eps_{perturb_seed}[g]),
 * bit-identical to es_restore(plan, restore_seed, sigma_restore) followed by
 * es_perturb(plan, perturb_seed, sigma_perturb): the intermediate value is
 * rounded to the storage type exactly as the separate calls would store it.
 * With restore_seed == perturb_seed (the two members of an antithetic pair,
 * sigma_perturb = -sigma_restore) the noise is generated once.
 * In the generation loop of §3 / App. D.6 the restore of member i and the
 * perturb of member i + 1 are adjacent (the next rollout follows the
 * perturb), so this halves the passes over the parameters in that loop.
 * Errors as es_perturb.
 */
es_status_t es_restore_perturb(es_plan_t plan, uint64_t restore_seed, float sigma_restore,
                               uint64_t perturb_seed, float sigma_perturb, void* stream);

/*
 * Fused reward-weighted update over the whole population in one pass (§3
 * implemented update; App. C.1):
 *   theta[g] <- round(theta[g] + sum_{i=0}^{n-1} coeffs[i] * eps_{seeds[i]}[g]),
 * the sum accumulated in fp32 in ascending i and rounded once to the storage
 * type, so theta is read and written exactly once. `seeds` and `coeffs` are
 * host arrays of length n (1 <= n <= ES_MAX_SEEDS). Seeds whose coefficient is
 * 0 are skipped; if every coefficient is 0 nothing is launched and theta stays
 * bit-identical (a batch with no valid reward leaves theta unchanged,
 * App. D.5/D.6).
 * Errors: ES_ERR_INVALID_ARG, ES_ERR_TOO_MANY_SEEDS, ES_ERR_NONFINITE,
 * ES_ERR_WRONG_DEVICE, ES_ERR_CUDA.
 */
es_status_t es_update(es_plan_t plan, const uint64_t* seeds, const float* coeffs,
                      int n, void* stream);

/*
 * The update of one generation fused with the first perturb of the next:
 *   theta[g] <- round(round(theta[g] + sum_i coeffs[i] * eps_{seeds[i]}[g])
 *                     + sigma_next * eps_{next_seed}[g]),
 * bit-identical to es_update(plan, seeds, coeffs, n) followed by
 * es_perturb(plan, next_seed, sigma_next), in one pass over theta. If every
 * coefficient is 0 this is es_perturb alone. Errors as es_update, and
 * ES_ERR_NONFINITE for sigma_next.
 */
es_status_t es_update_perturb(es_plan_t plan, const uint64_t* seeds, const float* coeffs,
                              int n, uint64_t next_seed, float sigma_next, void* stream);

/*
 * Replay of a logged run: the paper records the seed of every update and, for
 * evaluation, reloads the base checkpoint and reconstructs the update sequence
 * deterministically from those seeds (App. D.2, D.3, D.4). For g = 0 ..
 * generations-1, in order:
 *   theta[g] <- round(theta[g] + sum_{i in generation g} coeffs[i] * eps_{seeds[i]}[g]),
 * bit-identical to one es_update per generation. `seeds` and `coeffs` hold
 * the generations back to back; counts[g] (1 .. ES_MAX_SEEDS) is the size of
 * generation g. Generations of fewer than 4 non-zero seeds are fused, up to
 * 256 generations and ES_MAX_SEEDS seeds per pass over theta; a larger
 * generation gets a pass of its own, which computes it faster. Passes split
 * only between generations. Host arrays; asynchronous on `stream`. All arguments are
 * checked before the first pass; if a launch then fails (ES_ERR_CUDA), the
 * passes before it have been applied.
 * Errors: ES_ERR_INVALID_ARG (NULL, generations < 1, an empty generation),
 * ES_ERR_TOO_MANY_SEEDS (a generation over ES_MAX_SEEDS), ES_ERR_NONFINITE,
 * ES_ERR_WRONG_DEVICE, ES_ERR_CUDA.
 */
es_status_t es_replay(es_plan_t plan, const uint64_t* seeds, const float* coeffs,
                      const int* counts, int generations, void* stream);

/*
 * Population z-score of the rewards (§3):
 *   rhat_i = (R_i - mu) / (s + eps_z),  mu = (1/G) sum R_j,
 *   s^2 = (1/G) sum (R_j - mu)^2  (population variance).
 * A non-finite reward is first replaced by a finite penalty taken from the
 * batch itself, its smallest finite reward (the rule for invalid candidates of §5 and
 * App. D.5/D.6). If no reward is finite, or all are equal, every rhat_i is 0
 * (no update). Host-only. `rewards` and `rhat` may alias.
 * Errors: ES_ERR_INVALID_ARG (NULL, n < 1, eps_z < 0 or not finite).
 */
es_status_t es_normalize_rewards(const double* rewards, int n, double eps_z,
                                 double* rhat);

/*
 * Cosine schedule of sigma over the T generations (§3.1):
 *   sigma_t = sigma_T + (sigma_0 - sigma_T) (1 + cos(pi t / T)) / 2,
 * t clamped to [0, T]. Generation t = 0..T-1 uses sigma_t, so sigma_0 is used
 * first and sigma_T is the value after the last generation. T <= 0 returns
 * sigma_0. Host-only.
 */
double es_sigma_cosine(double sigma0, double sigmaT, int t, int T);

/*
 * Update coefficients c_i = alpha * rhat_i / (n * s), s = 1 for ES_SCALE_PAPER
 * and s = sigma for ES_SCALE_CANONICAL; computed in double, rounded once to
 * float. Host-only. Errors: ES_ERR_INVALID_ARG (NULL, n < 1, bad mode,
 * sigma <= 0 in canonical mode), ES_ERR_NONFINITE (a non-finite input or
 * result).
 */
es_status_t es_update_coeffs(const double* rhat, int n, double alpha, double sigma,
                             es_scale_t mode, float* coeffs);

/*
 * Antithetic pairs (not used by the paper, which is one-sided, App. D.5/D.6):
 * member (i,+) is evaluated at theta + sigma eps_i and member (i,-) at
 * theta - sigma eps_i. Both terms of the update share eps_i, so they fold into
 * one coefficient per seed:
 *   c_i = alpha * (rhat_pos[i] - rhat_neg[i]) / (2 * npairs * s),
 * with rhat normalised over all 2*npairs members and s as in es_update_coeffs.
 * Host-only. Errors as es_update_coeffs.
 */
es_status_t es_fold_antithetic(const double* rhat_pos, const double* rhat_neg,
                               int npairs, double alpha, double sigma,
                               es_scale_t mode, float* coeffs);

/*
 * Perturb without allocating. The paper has no counterpart to this entry
 * point; it exists for callers that must not allocate device memory after
 * start-up: a process whose device memory is handed out by its own pool or
 * caching allocator (a stray cudaMalloc there fragments memory the pool
 * counts as free, and cudaMalloc/cudaFree can synchronise the device), or a
 * latency-bound loop that may not call into the allocator at all.
 *
 * theta[g] <- round(theta[g] + sigma * eps_seed[g]) over the given segments,
 * exactly as es_perturb on a plan made from the same segments; pass -sigma to
 * restore. Segments follow the rules of es_plan_create (device memory of the
 * current device, 16-byte aligned data, index bases multiples of 8, no
 * overlap) and are validated on every call.
 *
 * Instead of a plan's table, the segment table is copied (cudaMemcpyAsync on
 * `stream`) into one static device array of ES_STATIC_MAX_SEGMENTS + 1
 * descriptors (about 32 KB), which every device that loads the library holds
 * until the process exits. The entry point calls no cudaMalloc, cudaFree or
 * other allocating routine, and uses about 36 KB of host stack.
 *   - More than ES_STATIC_MAX_SEGMENTS segments: ES_ERR_INVALID_ARG, nothing
 *     is launched.
 *   - All calls share the one array and each call rewrites it whole (nothing
 *     in it needs to start at zero); it keeps the last call's table. Calls
 *     that overlap on the GPU (on different streams, or from several host
 *     threads without ordering) race on that array and must not be issued.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current and keeps it for that
 *     device's context (after a device reset the next call looks it up
 *     again); make that first call before any stream capture.
 *   - A call on a stream that is being captured is refused with
 *     ES_ERR_INVALID_ARG before anything is copied or launched: the table is
 *     copied from the call's own stack, which a recorded copy would read again
 *     long after the call has returned.
 * Errors: ES_ERR_INVALID_ARG, ES_ERR_ALIGNMENT, ES_ERR_OVERLAP,
 * ES_ERR_NONFINITE, ES_ERR_CUDA.
 */
#define ES_STATIC_MAX_SEGMENTS 1024
es_status_t es_perturb_noalloc(const es_segment_t* segs, int nseg, es_dtype_t dtype,
                               uint64_t seed, float sigma, void* stream);

/* Static description of a status code. */
const char* es_status_string(es_status_t status);

/* Detail of the last error returned on the calling thread ("" if none). */
const char* es_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* ESOPT_H_ */
