// Internal declarations shared by the library's translation units (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace kvdro {

// Samples of one class are staged for the grid kernel as (x', x') float pairs, x' the sample plus
// the class's staging offset (stage_offset below), so that one 128-bit shared-memory load yields
// the packed operands of two samples.  Each class region starts on a multiple of kPadSamples and
// is padded with NaN pairs, which contribute exactly zero to the per-term kernels' excess sums
// (max(NaN, 0) = 0 in PTX max.f32 / max.f64); the exact kernel reads the padding as x = 0 and
// subtracts its known |0 - c| per cell.
constexpr int kPadSamples = 128;

// Error bits reported by kernels in ctx->d_err[1].
constexpr int kErrTimeout = 1;

struct SortArgs {
    const int32_t* lengths;     // caller samples (device), CSR by class
    const int64_t* offsets;     // [K+1]
    const int32_t* L;           // [K]
    const int64_t* hist_off;    // [K+1] start of class k's cumulative-count array (L_k + 1 entries)
    const int64_t* pair_off;    // [K+1] start of class k's padded pair region
    const int32_t* hist_blocks; // [K+1] prefix of histogram blocks per class
    const int32_t* exp_blocks;  // [K+1] prefix of expand blocks per class
    int32_t* hist;              // [hist_off[K]] counts, then cumulative counts (in place)
    int64_t* csum;              // [hist_off[K]] cumulative sums sum_{x <= v} x, or nullptr to skip
    int64_t* sumx;              // [K] sum of samples per class
    int32_t* sorted;            // [offsets[K]]
    float2* pairs;              // [pair_off[K]]
    int32_t* err;               // [0] += out-of-range samples
    int64_t* tile_tot;          // [K][scan_tiles][2] scan tile totals (count, sum of v h[v])
    int32_t* tile_lo;           // [exp_blocks[K] + K] per class from exp_blocks[k] + k: the bin of the
                                // first position of each expansion tile, then the bin of position N - 1
    int32_t scan_tiles;         // scan tiles of the largest class: ceil((max L + 1) / scan tile bins)
    int32_t K;
};

// Launchers (sort.cu)
// prefix[K + 1] of histogram blocks per class, sized to the current device (sort.cu)
cudaError_t hist_block_prefix(const int64_t* N, int32_t K, int32_t* prefix);
cudaError_t launch_histogram(const SortArgs& a, int32_t nblocks, cudaStream_t s);
cudaError_t launch_scan(const SortArgs& a, cudaStream_t s);
cudaError_t launch_expand(const SortArgs& a, int32_t nblocks, cudaStream_t s);
cudaError_t launch_gather_quantiles(const int32_t* sorted, const int64_t* offsets, const int32_t* rank, int32_t K,
                                    int32_t F, int32_t* out, cudaStream_t s);

// F32: per-term FP32 excess sums folded into FP64.  F64: per-term FP64.  EXACT: an exact integer
// threshold per cell, then per term an exact sum of |x - c| (packed FP32 adds and integer
// absolute differences side by side on two pipes), combined in FP64.
// ENVELOPE: the same sums in O(1) per cell from cumulative counts and sums (not per term).
enum class Prec { F32 = 0, F64 = 1, EXACT = 2, ENVELOPE = 3 };
constexpr int32_t kExactMaxL = 1 << 22;  // the exact kernel's integer sums need L <= 2^22

// Samples of a class whose support is at most kExactMaxL are staged as x + 2^23.  On [2^23, 2^24)
// a float's bit pattern is 0x4B000000 + x exactly, so the staged float serves both halves of the
// exact kernel without a conversion: packed FP32 adds on the value, integer absolute differences
// on the bits.  Larger supports are staged as x.  The FP32 and FP64 per-term kernels subtract
// the class's offset (exactly) from every sample.
constexpr float kStageOffset = 8388608.0f;  // 2^23
constexpr int32_t kStageBits = 0x4B000000;  // bit pattern of 2^23
__host__ __device__ inline float stage_offset(int32_t L) { return L <= kExactMaxL ? kStageOffset : 0.0f; }

struct GridArgs {
    const float2* pairs;        // padded (x', x') pairs, x' = x + stage_offset(L_k)
    const int64_t* pair_off;    // [K+1]
    const int64_t* N;           // [K]
    const int64_t* sumx;        // [K]
    const int32_t* L;           // [K]
    const int32_t* L_in;        // [K]
    const int32_t* cdf;         // cumulative counts, class k at hist_off[k]
    const int64_t* csum;        // cumulative sample sums, same layout (envelope mode)
    const int64_t* hist_off;    // [K+1]
    const int32_t* r;           // [R]
    const double* lam;          // [NL]
    const double* eps;          // [E]
    const double* cp;           // [M]
    const double* cw;           // [M]
    int32_t K, R, NL, E, M;
    int32_t LT;                 // lam tiles per CTA
    int32_t RG;                 // r groups per CTA
    int32_t r_blocks;           // CTAs per (m, k)
    int32_t m0, m_count;        // regime range covered by this launch
    int32_t f32_out;            // exact kernel: write S, cost and the argmin keys as FP32 (FP32 mode)
    void* S_out;                // optional [M][K][R][NL]
    void* cost_out;             // [M][E][K][R] (caller's, or scratch for FP64 min_cost)
    int32_t* lam_idx_out;       // optional [M][E][K][R]
    unsigned long long* keys;   // [M][E][K] argmin keys (initialised to all ones)
    int32_t* err;               // [1] |= kErrTimeout
    // Bounded waits and their test hook, per launch: wait_ns bounds each wait on a staged chunk
    // (0: the default of about 2 s); test_skip_chunk >= 0 leaves that chunk's copy unissued, so
    // the waits on it run out (-1 in production).
    long long wait_ns;
    int32_t test_skip_chunk;
    // Lam blocks: a grid of more lam values than one launch takes runs as consecutive launches over
    // blocks of it (ascending lam).  lam / NL are this block's values; lam0 is the index of its
    // first value in the caller's grid of NL_out values.  With several blocks, part_val / part_idx
    // ([m - m0][E][K][R]) carry each (r, eps) pair's minimum over the earlier blocks; the first
    // block starts them, the last writes the outputs.  One block: part_val is null, lam0 = 0.
    int32_t lam0, NL_out;
    double* part_val;
    int32_t* part_idx;
    int32_t part_first, part_last;
};

// The largest lam grid one launch of the exact kernel takes (16 warps of 2 x 8 tiles); larger
// grids run in blocks of it.
constexpr int32_t kExactLamBlock = 128;

struct FinalizeArgs {
    const unsigned long long* keys;
    const void* cost;           // FP64: cost buffer to read min_cost from; FP32 unused
    const int32_t* r;
    const int32_t* L_in;
    const int64_t* N;
    const int32_t* cdf;
    const int64_t* hist_off;
    int32_t K, R, E, M;
    int32_t* r_idx;             // [M][E][K]
    void* min_cost;             // [M][E][K]
    double* fhat;               // [M][E][K]
};

// grid.cu
// Launch shape of the grid kernel for one (precision, grid) problem: which compiled variant,
// lam tiles x r groups of warps per CTA, CTAs per (regime, class), dynamic shared memory.
struct GridShape {
    int variant;       // index of the compiled kernel instantiation
    int LT, RG;        // lam tiles and r groups per CTA
    int threads;       // 32 * LT * RG
    int r_blocks;      // CTAs per (m, k)
    size_t smem;
};
GridShape grid_shape(Prec p, int32_t R, int32_t NL, int32_t E, int32_t max_L);  // max_L: largest support
cudaError_t grid_prepare(Prec p);             // per-device attribute setup of every variant of p
// Launches over regimes [a.m0, a.m0 + a.m_count); fills a.LT, a.RG, a.r_blocks from `sh`.
cudaError_t launch_grid(Prec p, const GridShape& sh, GridArgs a, cudaStream_t s);
cudaError_t launch_finalize(Prec p, const FinalizeArgs& a, cudaStream_t s);

// dual.cu: exact minimisation over gamma >= 0 per (regime, radius, class, reservation)
struct DualArgs {
    const int32_t* cdf;         // cumulative counts, class k at hist_off[k]
    const int64_t* csum;        // cumulative sums, same layout
    const int64_t* hist_off;    // [K+1]
    const int64_t* N;           // [K]
    const int64_t* sumx;        // [K]
    const int32_t* L;           // [K]
    const int32_t* L_in;        // [K]
    const int32_t* r;           // [R]
    const double* eps;          // [E]
    const double* cp;           // [M]
    const double* cw;           // [M]
    int32_t K, R, E, M;
    double* cost;               // [M][E][K][R] (needed for min_cost)
    double* gamma;              // optional [M][E][K][R]
    unsigned long long* keys;   // [M][E][K], initialised to all ones
};
cudaError_t launch_dual(const DualArgs& a, cudaStream_t s);


#ifdef __CUDACC__
// The offset d = (c_p - mu) L - (c_p + c_w) eta of a cell's excess kappa x + d, evaluated as
// c_p (L - eta) - (mu L + c_w eta): L - eta is an exact integer and every product is rounded once,
// so a large c_p never swallows a small mu or c_w (the first form cancels to 0 at eta = L when
// mu and c_w are far below c_p, though d is then -(mu + c_w) L).  At the saturated multiplier
// mu = c_p the L terms vanish exactly and d = -(c_p + c_w) eta.  Every rounding is spelled out
// (no contraction left to the compiler), so each call site gets the same d bit for bit: a
// kernel that classifies samples twice at one multiplier (the dual's slope and value) must see
// the same threshold both times.
__device__ __forceinline__ double excess_offset(double cp, double cw, double mu, double L, double eta) {
    const double cw_eta = __dmul_rn(cw, eta);
    return mu == cp ? -__fma_rn(cp, eta, cw_eta) : __dsub_rn(__dmul_rn(cp, L - eta), __fma_rn(mu, L, cw_eta));
}

// The same excess about the reservation: kappa x + d = kappa (x - eta) + W(eta), with
//   W(eta) = (c_p - mu)(L - eta) - (c_w - nu) eta,
// for the per-term kernels, which add max(excess, 0) sample by sample.  x - eta is an exact
// integer; the two cost differences are exact or rounded once and each product is rounded once,
// so W(eta) is exactly 0 where the excess vanishes identically on one side of eta -- at the
// saturated multiplier (mu = c_p, nu = c_w), at eta = L with nu = c_w, at eta = 0 with mu = c_p --
// and a cell whose every term is zero sums to exactly zero.  (kappa x + d with the rounded d leaves
// the rounding error of mu L at x = L, which max(., 0) can pass on.)  The differences are at most
// the costs, so W(eta) is never less accurate than d.
__device__ __forceinline__ double excess_at_eta(double cp, double cw, double mu, double nu, double L, double eta) {
    return fma(__dsub_rn(cp, mu), L - eta, -__dmul_rn(__dsub_rn(cw, nu), eta));
}

// sum_n phi(x_n) with every sample on its own branch: V = c_w eta - nu x for the n - cnt samples
// below the cell's first active point, U = c_p (L - eta) - mu (L - x) for the cnt samples from it
// on.  The caller passes exact integer sums: sx_below = sum x below the point, dist_above =
// sum (L - x) from it on.  Nothing cancels beyond what each branch holds itself, whatever the
// ratios of c_p, c_w and the multiplier (V + max(U - V, 0) loses everything to cancellation
// when nu is many orders above the result).
// c i - m j for integers i, j held exactly in doubles: the rounding error of c i is recovered by
// one FMA, so the difference is rounded about once however closely the two products agree
// (forming both products first leaves only their rounding errors when they agree to 16 digits).
__device__ __forceinline__ double diff_of_products(double c, double i, double m, double j) {
    const double p = __dmul_rn(c, i);
    const double e = fma(c, i, -p);  // c i - p exactly, barring underflow
    return fma(-m, j, p) + e;
}

__device__ __forceinline__ double branch_sum(double cp, double cw, double mu, double nu, double L, double eta,
                                             double n, int64_t cnt, int64_t sx_below, int64_t dist_above) {
    return diff_of_products(cw, eta * (n - (double)cnt), nu, (double)sx_below) +
           diff_of_products(cp, (L - eta) * (double)cnt, mu, (double)dist_above);
}

// The per-term kernels sum phi as a base plus excesses: sum V + sum max(U - V, 0), or
// sum U + sum max(V - U, 0).  Each excess cancels, in the total, against the base's slope term
// (nu sum x, or mu sum (L - x)) on the samples it covers, so a cell takes the base whose slope
// is the smaller: U when nu > mu.  U - V = kappa x + d, so the U base negates kappa and d.
__device__ __forceinline__ bool use_u_split(double mu, double nu) { return nu > mu; }

// The first active support point of a cell: the smallest integer t in [0, L] with
// kappa * t + d > 0, or L + 1 when there is none (kappa >= 0, so the condition is monotone in
// t).  One FMA gives the sign of kappa * t + d exactly, so each test is exact.  An FP32 estimate
// of -d / kappa (off by a few units at most for L <= 2^24) is corrected by at most 8 such tests
// each way; should that not settle it, the FP64 quotient is corrected the same way.
__device__ __forceinline__ int64_t first_active(double kappa, double d, int64_t L) {
    if (d > 0.0) return 0;
    if (!(kappa > 0.0) || !(fma(kappa, (double)L, d) > 0.0)) return L + 1;
    // here t is in [1, L]: kappa (t - 1) + d <= 0 < kappa t + d
    auto settle = [&](double q, int64_t& t) {
        const double e = floor(q) + 1.0;
        t = e < 1.0 ? 1 : (e > (double)L ? L : (int64_t)e);
        for (int i = 0; i < 8 && t > 1 && fma(kappa, (double)(t - 1), d) > 0.0; i++) t--;
        for (int i = 0; i < 8 && t < L && !(fma(kappa, (double)t, d) > 0.0); i++) t++;
        return (t == 1 || !(fma(kappa, (double)(t - 1), d) > 0.0)) && fma(kappa, (double)t, d) > 0.0;
    };
    int64_t t;
    if (settle((double)__fdiv_rn(-(float)d, (float)kappa), t)) return t;
    (void)settle(-d / kappa, t);
    return t;
}
#endif

}  // namespace kvdro
