/*
 * kvdro.h -- C ABI of the GB300 Wasserstein-DRO KV-reservation grid evaluator.
 *
 * The library evaluates, on one GPU, the worst-case expected reservation cost
 * of the paper "Robust KV Cache Management for LLM Serving under Output Token
 * Length Uncertainty" over a grid of
 *     regimes m (a (c_p, c_w) pair) x classes k x reservations r x multipliers lam x radii eps
 * and reduces it to a per-(regime, radius, class) reservation.  For class k with
 * samples x_1..x_N (output lengths in tokens), support [0, L_k] and input
 * length L_in_k, with eta = r - L_in_k:
 *
 *   Q(eta, xi)   = c_p (xi - eta)^+ + c_w (eta - xi)^+                 (Sec. 2.3; App. A Step 1)
 *   phi_n        = max{ Q(eta,0) - lam x_n, Q(eta,x_n), Q(eta,L) - lam (L - x_n) }
 *                                                                       (App. A Step 4)
 *   S(eta, lam)  = (1/N) sum_n phi_n                                   (App. A Step 3)
 *   cost(eta,eps)= min_j ( lam_j eps + S(eta, lam_j) )                 (App. A eq. app_kantorovich,
 *                                                                        gamma restricted to the lam grid)
 *   r*           = argmin_r cost                                        (Sec. 2.4, eq. dro_obj, r block)
 *   quantiles    = lower empirical quantiles x_(max(1, ceil(q N)))     (Prop. "Critical Fractile
 *                                                                        Structure", eq. critical_fractile)
 *
 * Conventions shared by every entry point
 *   - Every function returns a kvdro_status.  Nothing is thrown or aborted across the ABI.
 *   - Argument errors are found on the host before any launch (KVDRO_EINVAL) and leave the
 *     context unchanged; kvdro_last_error() then describes the error.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = the legacy default stream).
 *     Asynchronous CUDA errors surface at the next call or at kvdro_sync() (KVDRO_ECUDA).
 *   - Array arguments marked "host or device" may point to either; the library inspects the
 *     pointer.  When any such OUTPUT is in host memory the call blocks until it is filled.
 *     Device outputs are written asynchronously on `stream`.
 *   - The caller owns every buffer it passes; the library owns only what it allocates inside the
 *     context (the loaded samples' sorted copies and cumulative arrays, and the staging and scratch
 *     of the evaluation calls, kept for reuse), and kvdro_destroy() frees that.
 *   - A context belongs to one device and one host thread at a time.
 *   - Ties: the minimum over lam and the argmin over r both take the lowest index.
 */
#ifndef KVDRO_H
#define KVDRO_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct kvdro_ctx kvdro_ctx;

typedef enum {
    KVDRO_OK = 0,
    KVDRO_EINVAL = -1,   /* bad argument; nothing was launched */
    KVDRO_ENOMEM = -2,   /* a device or pinned-host allocation failed */
    KVDRO_ECUDA = -3,    /* a CUDA call failed (message in kvdro_last_error) */
    KVDRO_ESTATE = -4,   /* call out of order, e.g. eval before samples are loaded */
    KVDRO_ETIMEOUT = -5  /* a kernel gave up a bounded wait and reported it */
} kvdro_status;

typedef enum {
    KVDRO_FP32 = 0,      /* FP32 outputs.  When every L_max <= 2^22 they are the KVDRO_EXACT
                            results rounded to FP32 (the exact kernel is also the fastest);
                            otherwise per-term arithmetic in FP32 with sums folded into FP64 */
    KVDRO_FP64 = 1,      /* per-term arithmetic and sums in FP64 */
    KVDRO_EXACT = 2,     /* per term, exact integer arithmetic on exact integer thresholds
                            (|x + 1 - t| summed exactly, half of the cells in packed FP32 adds,
                            half in integer absolute differences); exact integer counts and
                            sums combined once per cell in FP64, so results carry FP64 rounding
                            only.  Needs every L_max <= 2^22. */
    KVDRO_ENVELOPE = 3   /* not per term: each cell's sample sum from the sorted samples'
                            cumulative counts and sums at its exact threshold, O(1) per cell,
                            FP64 outputs with FP64 rounding only */
} kvdro_precision;

/* Create a context on CUDA device `device_ordinal`.  *out receives the handle (NULL on error).
 * Two environment variables, read here, are test hooks and must not be set in production:
 * KVDRO_TEST_FAIL_ALLOC=n makes the context's n-th allocation fail (KVDRO_ENOMEM), and
 * KVDRO_TEST_SKIP_CHUNK=c makes this context's grid kernels leave staged chunk c uncopied with a
 * wait bound of 1 ms, so every bounded wait on it runs out (KVDRO_ETIMEOUT).  The hook travels
 * with this context's launches only; other contexts, on the same device or not, keep the
 * production bound.
 * Bounded waits: a grid kernel gives up waiting for a staged sample chunk only after 2 s of the
 * GPU's global timer AND a minimum number of polls made while it was running, so a CTA that is
 * descheduled (time-slicing, preemption) does not report a timeout on a copy that lands once it
 * resumes. */
int kvdro_create(kvdro_ctx** out, int device_ordinal);

/*
 * Load the per-class empirical samples (the empirical distribution of Sec. 2.4 and the
 * Alg. 1 input) and sort them.  Replaces any previously loaded samples.
 *   K        number of classes, 1 <= K <= 4096.
 *   offsets  host int64[K+1], CSR offsets: offsets[0] = 0, N_k = offsets[k+1] - offsets[k] >= 1,
 *            N_k <= 2^31 - 1.
 *   lengths  host or device int32[offsets[K]], class k's samples at [offsets[k], offsets[k+1]),
 *            each in [0, L_max[k]] (checked on the device; a violation gives KVDRO_EINVAL).
 *   L_max    host int32[K], support upper end L_k, 1 <= L_k <= 2^24.
 *   L_in     host int32[K] input length per class (>= 0, L_in + L_max <= 2^24), or NULL for zeros.
 * Runs the segmented counting sort and the cumulative count arrays on `stream`, then blocks
 * until the range check has been read back.
 */
int kvdro_load_samples(kvdro_ctx* ctx, int32_t K, const int64_t* offsets, const int32_t* lengths,
                       const int32_t* L_max, const int32_t* L_in, void* stream);

/*
 * Lower empirical quantiles of every loaded class: out[k*F + f] = x_(m), the m-th smallest
 * sample of class k, m = max(1, ceil(fractiles[f] * N_k)) computed in FP64.
 *   F          1 <= F <= 65536;  fractiles: host double[F], each in [0, 1].
 *   out        host or device int32[K*F].
 */
int kvdro_quantiles(kvdro_ctx* ctx, int32_t F, const double* fractiles, int32_t* out, void* stream);

/*
 * Evaluate the grid and reduce it.  Element type of S, cost and min_cost is float for
 * KVDRO_FP32 and double for the other modes.
 *   R, r       host int32[R], 1 <= R <= 2^20; every r must satisfy L_in_k <= r <= L_in_k + L_k for
 *              every class (the reservation domain of Sec. 2.2).
 *   NL, lam    host double[NL], finite, >= 0; 1 <= NL <= 256 (128 for KVDRO_FP64).  The exact
 *              kernel (KVDRO_EXACT, and KVDRO_FP32 when every L_max <= 2^22) takes 128 lam values
 *              per launch; a larger grid runs as consecutive launches over blocks of 128 with the
 *              running minimum in context scratch (12 bytes per (regime, eps, class, r), at most
 *              256 MB at a time).
 *   E, eps     host double[E], finite, >= 0; 1 <= E <= 64.
 *   M, c_p,c_w host double[M] each, finite, >= 0; 1 <= M <= 65536.
 * Outputs (each may be NULL to skip it; host or device).  With M > 1, host S, cost and lam_idx
 * come back in up to 16 blocks of regimes on a stream of the context's own; into page-locked host
 * memory each block's copy overlaps the evaluation of the next (a copy into pageable memory holds
 * the calling thread until it is done, so those blocks alternate with the evaluation instead).
 * The call returns only once every output is filled.
 *   S          [M][K][R][NL]  mean supremum S(eta, lam)
 *   cost       [M][E][K][R]   min over lam of lam*eps + S
 *   lam_idx    int32 [M][E][K][R]  lowest lam index attaining cost
 *   r_idx      int32 [M][E][K]     lowest r index attaining min_r cost
 *   min_cost   [M][E][K]
 *   fhat       double [M][E][K]    #{x <= r* - L_in} / N  (empirical CDF at the chosen r)
 */
int kvdro_eval_grid(kvdro_ctx* ctx, int precision, int32_t R, const int32_t* r, int32_t NL, const double* lam,
                    int32_t E, const double* eps, int32_t M, const double* c_p, const double* c_w, void* S,
                    void* cost, int32_t* lam_idx, int32_t* r_idx, void* min_cost, double* fhat, void* stream);

/*
 * The exact worst-case expected cost, without restricting gamma to a grid: for every regime,
 * radius, class and reservation, min over gamma >= 0 of gamma*eps + S(eta, gamma) (App. A,
 * eq. app_kantorovich; the value of the epigraph LP of eq. app_lp, which equals the worst case
 * over the Wasserstein ball by the strong duality of App. A Step 2).  The objective is convex
 * and piecewise linear in gamma with its minimiser in [0, max(c_p, c_w)]; the library bisects on
 * its right derivative over the ordered bit patterns of the nonnegative doubles (at most 63
 * steps, down to two adjacent doubles at any scale) with every evaluation O(1) from the sorted
 * samples' cumulative counts and sums, so results carry FP64 rounding only.  The result is
 * never below the empirical cost (1/N) sum_n Q(eta, x_n), computed exactly from integer sums:
 * that bound holds at every gamma (App. A) and is the value itself at eps = 0.
 * Arguments as kvdro_eval_grid; outputs (each may be NULL; host or device):
 *   cost       double [M][E][K][R]   the exact dual value
 *   gamma      double [M][E][K][R]   a minimising gamma
 *   r_idx      int32 [M][E][K]       lowest r index attaining the minimum (among costs equal to
 *                                    2^-32 relative)
 *   min_cost   double [M][E][K];  fhat  double [M][E][K]  as in kvdro_eval_grid
 */
int kvdro_eval_dual(kvdro_ctx* ctx, int32_t R, const int32_t* r, int32_t E, const double* eps, int32_t M,
                    const double* c_p, const double* c_w, double* cost, double* gamma, int32_t* r_idx,
                    double* min_cost, double* fhat, void* stream);

/* Copy the sorted samples (class by class, ascending, int32[offsets[K]]) to `out` (host or device). */
int kvdro_sorted_samples(const kvdro_ctx* ctx, int32_t* out, void* stream);

/*
 * Device time, in milliseconds, of the grid-kernel launches of the last kvdro_eval_grid() or
 * kvdro_eval_dual() call on this context, measured with CUDA events recorded on that call's
 * stream immediately before and after them (the argmin finalisation and the output copies are
 * outside).  Blocks until the second event has completed.  KVDRO_ESTATE if nothing has been
 * evaluated yet.
 */
int kvdro_last_grid_ms(kvdro_ctx* ctx, float* ms);

/*
 * kvdro_eval_grid_noalloc -- the FP32 grid evaluation (load, sort, grid, argmin) in one call
 * that allocates nothing.  The paper has no counterpart; this entry point exists for callers
 * that cannot allocate device memory at the time they need an answer: a serving engine that
 * has handed all free device memory to its KV-cache block pool at start-up (a new cudaMalloc
 * would fail or evict cache blocks), a process held to a fixed device-memory budget, or a
 * latency-critical loop that must not call cudaMalloc/cudaFree because cudaFree synchronises
 * the whole device.
 *
 * Instead of a context, it works in one static device array of KVDRO_NOALLOC_SCRATCH_BYTES
 * bytes, defined in the library; every GPU that loads the library holds that array until the
 * process exits.  The first call on a device (with that device current) resolves the array's
 * device address and sets a kernel attribute; make that first call before any stream capture.
 * Calls share the array: it keeps the last call's contents (the call clears what must start at
 * zero), and calls whose GPU work overlaps in time race on it -- serialise them, e.g. on one
 * stream.  A problem whose scratch would exceed the array (about 12 bytes per sample plus
 * 4 bytes per support point and 8 bytes per (regime, radius, class) row, and with more than 128
 * lam values 12 bytes per (regime, radius, class, r) cell) is rejected with KVDRO_EINVAL and a
 * message.
 *
 * Arguments are those of kvdro_load_samples and kvdro_eval_grid with precision KVDRO_FP32,
 * on the current device, except that `lengths` and every output must be device memory, there
 * is no S output, and `err` (may be NULL) receives up to err_len bytes of error text.  The
 * call works on `stream` and returns once the outputs are written (it reads the samples' range
 * check and the kernels' status word back), so a grid kernel that gave up a bounded wait is
 * reported here as KVDRO_ETIMEOUT (the outputs are then incomplete).  The test hook
 * KVDRO_TEST_SKIP_CHUNK of kvdro_create is read at every call of this entry point.
 */
#define KVDRO_NOALLOC_SCRATCH_BYTES (32u << 20)
int kvdro_eval_grid_noalloc(int32_t K, const int64_t* offsets, const int32_t* lengths, const int32_t* L_max,
                            const int32_t* L_in, int32_t R, const int32_t* r, int32_t NL, const double* lam,
                            int32_t E, const double* eps, int32_t M, const double* c_p, const double* c_w,
                            float* cost, int32_t* lam_idx, int32_t* r_idx, float* min_cost, double* fhat,
                            void* stream, char* err, int32_t err_len);

/* Wait for the context's device work and report any asynchronous CUDA error or kernel timeout. */
int kvdro_sync(kvdro_ctx* ctx);

/* Text of the last error on this context ("" if none).  Valid until the next call on ctx. */
const char* kvdro_last_error(const kvdro_ctx* ctx);

/* Free the context and everything it owns.  NULL is accepted. */
int kvdro_destroy(kvdro_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* KVDRO_H */
