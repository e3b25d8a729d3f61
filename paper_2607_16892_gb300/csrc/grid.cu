// Grid evaluation of the worst-case reservation cost (the hot path) and its reductions.
//
// What is summed.  For class k (samples x_n in [0, L], count N), regime (c_p, c_w), reservation
// r with eta = r - L_in in [0, L], and multiplier lam >= 0, the per-sample supremum of App. A
// Step 4 is the maximum of four affine functions of x:
//   l1 = c_p (x - eta), l2 = c_w (eta - x)            (the two branches of Q(eta, x))
//   l3 = Q(eta, 0) - lam x = c_w eta - lam x          (sample moved to xi = 0)
//   l4 = Q(eta, L) - lam (L - x) = c_p (L - eta) - lam (L - x)   (moved to xi = L)
// Since l3 - l2 = (c_w - lam) x and l4 - l1 = (c_p - lam)(L - x), with x and L - x >= 0:
//   max(l2, l3) = V(x) = c_w eta - nu x,           nu = min(lam, c_w)
//   max(l1, l4) = U(x) = c_p (L - eta) - mu (L - x),  mu = min(lam, c_p)
// so phi = max(U, V) = V + max(W, 0) with W = U - V = kappa x + d,
//   kappa = mu + nu,   d = (c_p - mu) L - (c_p + c_w) eta.
// Summing over the class: sum_n phi_n = N c_w eta - nu sum_n x_n + sum_n max(kappa x_n + d, 0).
// Three forms of that sum:
//  - FP32 and FP64 per term: the excess max(kappa x + d, 0) term by term on the base V, or
//    max(-(kappa x + d), 0) on the base U when nu > mu, whichever cancels less (use_u_split).  The
//    excess is evaluated about the reservation, kappa (x - eta) + W(eta) (excess_at_eta), so that
//    it is exactly zero wherever it vanishes identically on one side of eta.  FP64: one fused
//    multiply-add, one max and one add per sample and cell.  FP32: one saturating fused
//    multiply-add on the excess scaled by a power of two (the clamp to [0, 1] is the max) and half
//    a packed add per sample and cell.
//  - EXACT (also FP32 requests whose supports are all <= 2^22): each cell's integer threshold t
//    (x >= t exactly when kappa x + d > 0), then per term the exact sum of |x + 1 - t|, half of a
//    warp's cells on packed FP32 adds and half on integer absolute differences, so the FMA and ALU
//    pipes work side by side; the epilogue puts every sample on its own branch (branch_sum).
//  - ENVELOPE (k_envelope): the same branch sums from the cumulative counts and sums, O(1) per
//    cell, not per term.
//
// Work decomposition.  A CTA owns one (regime m, class k) and a block of RG*TR consecutive r
// values for the whole lam grid.  Each warp owns a TR x TL tile of (r, lam) cells; its 32 lanes
// split the class's samples, which stream through a ring of shared-memory chunks filled by TMA
// bulk copies (cp.async.bulk + mbarrier).  Packed f32x2 instructions serve two cells at once.
// Periodically each lane's partial sums are transposed and reduced across the warp (fixed
// shuffle order) so that each lane then owns one cell, folded into an FP64 or int64 accumulator.
// The epilogue forms S = (1/N) sum phi, then for every eps the minimum over lam (lowest index),
// and feeds the argmin over r through a 64-bit atomicMin on (cost, r index) keys.
#include <float.h>
#include <math.h>

#include "kvdro_internal.cuh"

namespace kvdro {
namespace {

typedef unsigned long long u64;

// Bound on any barrier wait: 2 s of the GPU's global nanosecond timer, and at least
// kWaitPollsPerNs polls per nanosecond of that bound spent polling (each poll suspends the
// thread for at most kPollSuspendNs).  The timer keeps running while a CTA is descheduled
// (time-slicing, preemption), but the poll count only grows while it runs, so a CTA that
// was switched out for longer than the bound does not give up on a copy that lands soon
// after it resumes.  kWaitPollCap bounds the loop even if the timer were to stop.
constexpr long long kWaitNs = 2000000000LL;
constexpr unsigned kPollSuspendNs = 1000;
constexpr long long kWaitNsPerPoll = 4096;   // polls required: limit_ns / 4096
constexpr unsigned kWaitPollCap = 1u << 28;

constexpr int ilog2(int v) { return v <= 1 ? 0 : 1 + ilog2(v / 2); }

// Shape of one instantiation of the grid kernel: precision, warp tile (TR reservations x TL
// multipliers, TR*TL a power of two <= 32), FP32 chunks between folds of the per-lane partial
// sums into FP64 (FP64 folds once at the end), the largest CTA and minimum CTAs per SM it is
// compiled for (these two bound its registers per thread), the staged chunk and ring depth, the
// sample loop's unroll, and (exact) the lam columns per row on packed FP32 adds.
template <Prec P_, int TR_, int TL_, int FLUSH_, int MINB_, int MAXT_ = 512, int CHUNK_ = 2048, int STAGES_ = 3,
          int UNROLL_ = 2, int FCOLS_ = TL_ / 2>
struct GridCfg {
    static constexpr int FCOLS = FCOLS_;
    static constexpr Prec P = P_;
    static constexpr int TR = TR_, TL = TL_, V = TR_ * TL_, LOG2V = ilog2(TR_ * TL_), FLUSH = FLUSH_, MINB = MINB_;
    static constexpr int MAXT = MAXT_;
    static constexpr int CHUNK = CHUNK_;    // samples per staged chunk (float2 each)
    static constexpr int STAGES = STAGES_;  // ring depth
    static constexpr int UNROLL = UNROLL_;  // unroll of the sample loop
    static_assert(CHUNK_ % 128 == 0 && CHUNK_ * 8 * STAGES_ <= 160 * 1024, "chunk ring must fit shared memory");
    static_assert((V & (V - 1)) == 0 && V >= 2 && V <= 32, "tile must hold a power of two <= 32 cells");
    static_assert(P_ == Prec::F64 || TL_ % 2 == 0, "the FP32 and exact tiles pack lam values in pairs");
    static_assert(FLUSH >= 0 && UNROLL >= 1 && FCOLS >= 0 && FCOLS <= TL, "shape parameters out of range");
};
// 2 r x 8 lam tiles, up to 16 warps per CTA and (FP32, exact) two CTAs per SM (64 registers)
// for up to 128 lam values; larger lam grids run the exact kernel in blocks of 128 lam values
// (kExactLamBlock), and the FP32 kernel takes 2 x 16 tiles.  FP64: 2 x 8 tiles.
// The exact variants stage 6144-sample chunks (48 KB), the FP32 and FP64 ones 4096-sample chunks
// (32 KB), through a 2-deep ring (two CTAs of the exact kernel per SM: 2 x 96 KB of ring).  The FP32
// variants fold their partial sums every 2 chunks (256 samples per lane); the exact variants fold
// as often as their support size requires, independently of the chunk size.  The FP32 and exact
// variants unroll the sample loop 4 times, and the exact variants give half of every row's lam
// columns (FCOLS) to the packed FP32 adds, the rest to the integer absolute differences.
using CfgF32 = GridCfg<Prec::F32, 2, 8, 2, 2, 512, 4096, 2, 4>;
using CfgF32Wide = GridCfg<Prec::F32, 2, 16, 2, 1, 512, 4096, 2, 4>;
using CfgF64 = GridCfg<Prec::F64, 2, 8, 0, 1, 512, 4096, 2>;
using CfgExact = GridCfg<Prec::EXACT, 2, 8, 0, 2, 512, 6144, 2, 4>;
// Above a support of 2^19 the packed FP32 sums (exact only up to 2^24) would fold every few loads;
// there every column takes the integer absolute differences, whose sums fold far less often.
using CfgExactInt = GridCfg<Prec::EXACT, 2, 8, 0, 2, 512, 6144, 2, 8, 0>;
// One or two lam values (a small grid, or the last block of a larger one): 8 r x 2 lam tiles, so
// that a single value pads its tile to 2 columns rather than 8; both columns on the integer sad.
using CfgExactFewLam = GridCfg<Prec::EXACT, 8, 2, 0, 2, 512, 6144, 2, 8, 0>;
constexpr int32_t kFewLam = 2;
constexpr int32_t kExactIntAboveL = 1 << 19;
constexpr int kWarpsTarget = 16;  // warps per CTA the r groups fill up to
static_assert(kExactLamBlock == kWarpsTarget * CfgExact::TL && kExactLamBlock == kWarpsTarget * CfgExactInt::TL,
              "one launch of the exact kernel takes 16 warps of lam tiles");

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ u64 pk(float lo, float hi) {
    u64 r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void upk(u64 r, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(r));
}
__device__ __forceinline__ u64 fadd2(u64 a, u64 b) {
    u64 r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
// a b + c rounded once, then clamped to [0, 1]; a NaN result becomes 0.  For |a b + c| <= 1 this is
// max(a b + c, 0) in one instruction on the FMA pipe.
__device__ __forceinline__ float fma_sat(float a, float b, float c) {
    float d;
    asm("fma.rn.sat.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ u64 abs2(u64 v) {
    float a, b;
    upk(v, a, b);
    return pk(fabsf(a), fabsf(b));
}
// max(w, 0); a NaN operand yields 0 (PTX max returns the non-NaN input).
__device__ __forceinline__ double relu(double w) {
    double d;
    asm("max.f64 %0, %1, 0d0000000000000000;" : "=d"(d) : "d"(w));
    return d;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// One bulk copy global -> shared, completing on `bar` (bytes and both addresses 16-byte aligned).
__device__ __forceinline__ void tma_bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// The same test, suspending the thread for at most about `ns` nanoseconds while the phase is
// incomplete.
__device__ __forceinline__ bool mbar_try_for(uint32_t bar, uint32_t parity, uint32_t ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(ns)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait for phase `parity` of `bar`.  Gives up and returns false once limit_ns nanoseconds of
// the global timer have passed and the wait has polled at least limit_ns / kWaitNsPerPoll
// times (or after kWaitPollCap polls in any case).  limit_ns <= 0 selects kWaitNs.
__device__ __noinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, long long limit_ns) {
    if (mbar_try(bar, parity)) return true;
    if (limit_ns <= 0) limit_ns = kWaitNs;
    const unsigned long long t0 = global_ns();
    const unsigned min_polls = (unsigned)(limit_ns / kWaitNsPerPoll);
    unsigned polls = 0;
    while (!mbar_try_for(bar, parity, kPollSuspendNs)) {
        ++polls;
        if (polls >= kWaitPollCap) return false;
        if (polls >= min_polls && (long long)(global_ns() - t0) > limit_ns) return false;
    }
    return true;
}

// Reduce V per-lane values across the warp so that lane l ends with the warp-wide sum of value
// index l >> (5 - log2 V): recursive halving over lane bits 4, 3, ..., then butterflies over the
// remaining low bits.  The order of additions is fixed, so results are deterministic.
template <typename T, int V, int S>
struct TransposeStep {
    static __device__ __forceinline__ void run(T (&v)[V], int lane) {
        constexpr int n = V * S / 16;  // values still held per lane before this step
        if constexpr (n >= 2) {
            constexpr int h = n / 2;
            const bool up = (lane & S) != 0;
#pragma unroll
            for (int p = 0; p < h; p++) {
                const T send = up ? v[p] : v[p + h];
                const T keep = up ? v[p + h] : v[p];
                v[p] = keep + __shfl_xor_sync(0xffffffffu, send, S);
            }
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], S);
        }
        if constexpr (S > 1) TransposeStep<T, V, S / 2>::run(v, lane);
    }
};

template <typename T, int V>
__device__ __forceinline__ T transpose_reduce(T (&v)[V], int lane) {
    TransposeStep<T, V, 16>::run(v, lane);
    return v[0];
}

struct SmemLayout {
    size_t ring, full, lam, eps, S, total;
};

__host__ __device__ inline SmemLayout smem_layout(int RG, int TR, int NLpad, int E, int chunk, int stages) {
    SmemLayout L;
    L.ring = 0;
    L.full = (size_t)stages * chunk * sizeof(float2);
    L.lam = L.full + 8 * (size_t)stages;
    L.eps = L.lam + 8 * (size_t)NLpad;
    L.S = L.eps + 8 * (size_t)E;
    L.total = L.S + 8 * (size_t)RG * TR * NLpad;
    return L;
}

// Epilogue of one CTA: for each of its (r, eps) pairs, the minimum over lam of lam * eps + S
// (lowest index on ties), the cost and lam index outputs, and the argmin over r through a 64-bit
// atomicMin key (FP32: cost bits and r index; otherwise the cost's double bits truncated to 44
// bits, order-preserving for non-negative values, with the r index in the low 20 bits).
template <bool F32OUT>
__device__ __forceinline__ void cta_epilogue(const GridArgs& a, const double* s_S, const double* s_lam,
                                             const double* s_eps, int stride, int rl_count, int r_cta0, int m, int k) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    for (int p = warp; p < rl_count * a.E; p += nwarps) {
        const int rl = p / a.E, e = p % a.E;
        const int ri = r_cta0 + rl;
        if (ri >= a.R) continue;
        double best = DBL_MAX;
        int bj = 0x7fffffff;
        for (int j = lane; j < a.NL; j += 32) {
            const double v = __dadd_rn(__dmul_rn(s_lam[j], s_eps[e]), s_S[rl * stride + j]);
            if (v < best) { best = v; bj = j; }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const double ov = __shfl_xor_sync(0xffffffffu, best, o);
            const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
            if (ov < best || (ov == best && oj < bj)) { best = ov; bj = oj; }
        }
        if (lane == 0) {
            const size_t row = ((size_t)m * a.E + e) * a.K + k;
            const size_t o = row * a.R + ri;
            bj += a.lam0;
            if (a.part_val) {  // lam blocks: merge with the earlier blocks (they hold lower indices)
                const size_t q = ((((size_t)(m - a.m0)) * a.E + e) * a.K + k) * a.R + ri;
                if (!a.part_first && !(best < a.part_val[q])) {
                    best = a.part_val[q];
                    bj = a.part_idx[q];
                }
                if (!a.part_last) {
                    a.part_val[q] = best;
                    a.part_idx[q] = bj;
                    continue;
                }
            }
            u64 key;
            if constexpr (F32OUT) {
                const float cf = (float)best;
                if (a.cost_out) static_cast<float*>(a.cost_out)[o] = cf;
                key = ((u64)__float_as_uint(cf > 0.f ? cf : 0.f) << 32) | (u64)(uint32_t)ri;
            } else {
                static_cast<double*>(a.cost_out)[o] = best;
                key = ((u64)__double_as_longlong(best > 0.0 ? best : 0.0) & ~0xFFFFFull) | (u64)ri;
            }
            if (a.lam_idx_out) a.lam_idx_out[o] = bj;
            atomicMin(a.keys + row, key);
        }
    }
}

// ---------------------------------------------------------------- the grid kernel

template <class C>
__global__ void __launch_bounds__(C::MAXT, C::MINB) k_grid(const GridArgs a) {
    constexpr Prec P = C::P;
    constexpr int TR = C::TR, TL = C::TL, V = C::V, LOG2V = C::LOG2V;
    extern __shared__ __align__(128) unsigned char smem[];
    const int NLpad = a.LT * TL;
    const SmemLayout lay = smem_layout(a.RG, TR, NLpad, a.E, C::CHUNK, C::STAGES);
    float2* ring = reinterpret_cast<float2*>(smem + lay.ring);
    u64* full = reinterpret_cast<u64*>(smem + lay.full);
    double* s_lam = reinterpret_cast<double*>(smem + lay.lam);
    double* s_eps = reinterpret_cast<double*>(smem + lay.eps);
    double* s_S = reinterpret_cast<double*>(smem + lay.S);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    int b = blockIdx.x;
    const int rb = b % a.r_blocks;
    b /= a.r_blocks;
    const int k = b % a.K;
    const int m = a.m0 + b / a.K;
    const int lt = warp % a.LT, rg = warp / a.LT;
    const int r_cta0 = rb * a.RG * TR;
    const int r_local0 = rg * TR;

    for (int i = tid; i < NLpad; i += blockDim.x) s_lam[i] = i < a.NL ? a.lam[i] : 0.0;
    for (int i = tid; i < a.E; i += blockDim.x) s_eps[i] = a.eps[i];

    const int64_t pbase = a.pair_off[k];
    const int64_t np = a.pair_off[k + 1] - pbase;  // multiple of kPadSamples
    const int nchunks = (int)((np + C::CHUNK - 1) / C::CHUNK);
    const float2* src = a.pairs + pbase;
    auto issue = [&](int c) {
        if (c == a.test_skip_chunk) return;  // test hook: nothing will complete this chunk's barrier
        const int s = c % C::STAGES;
        const int64_t cnt = min((int64_t)C::CHUNK, np - (int64_t)c * C::CHUNK);
        tma_bulk_load(smem_u32(ring + (size_t)s * C::CHUNK), src + (int64_t)c * C::CHUNK, (uint32_t)(cnt * sizeof(float2)),
                      smem_u32(&full[s]));
    };
    __shared__ double s_inv_n;  // 1 / N, one FP64 division per CTA (FP64 runs at 1/64 of FP32 here)
    if (tid == 0) {
        for (int s = 0; s < C::STAGES; s++) mbar_init(smem_u32(&full[s]), 1);
        fence_mbar_init();
        s_inv_n = 1.0 / (double)a.N[k];
    }
    __syncthreads();
    if (tid == 0)
        for (int c = 0; c < C::STAGES && c < nchunks; c++) issue(c);
    int issued = min(C::STAGES, nchunks);  // chunks issued so far (tracked identically by every thread)
    int consumed = 0;                    // chunk at which the loop stopped

    // Per-cell constants of this warp's tile (identical across its lanes).
    const double cp = a.cp[m], cw = a.cw[m], Lk = (double)a.L[k];
    double eta[TR];
    bool rvalid[TR];
#pragma unroll
    for (int i = 0; i < TR; i++) {
        const int ri = r_cta0 + r_local0 + i;
        rvalid[i] = ri < a.R;
        eta[i] = rvalid[i] ? (double)a.r[ri] - (double)a.L_in[k] : 0.0;
    }

    bool timeout = false;
    double acc64 = 0.0;  // this lane's cell after the warp transposition

    if constexpr (P == Prec::F32) {
        // Each row's excess is taken about its reservation: kappa (x - eta) + W(eta) (excess_at_eta).
        // x - eta comes from the staged samples in one packed add per row and load (both samples of
        // the load): the staged value carries the class's offset, and offset + eta is an integer
        // below 2^24, so the add is exact.
        const double offd = (double)stage_offset(a.L[k]);
        u64 noff[TR];
#pragma unroll
        for (int i = 0; i < TR; i++) {
            const float o = (float)-(offd + eta[i]);
            noff[i] = pk(o, o);
        }
        u64 kap[TL / 2], dd[TR][TL / 2], acc[TR][TL / 2];
#pragma unroll
        for (int jp = 0; jp < TL / 2; jp++) {
            const int j0 = lt * TL + 2 * jp;
            const double l0 = s_lam[j0], l1 = s_lam[j0 + 1];
            const bool v0 = j0 < a.NL, v1 = j0 + 1 < a.NL;
            const double mu0 = fmin(l0, cp), mu1 = fmin(l1, cp), nu0 = fmin(l0, cw), nu1 = fmin(l1, cw);
            // the split of phi this column sums (see use_u_split): the sign of its excess
            const float s0 = use_u_split(mu0, nu0) ? -1.f : 1.f, s1 = use_u_split(mu1, nu1) ? -1.f : 1.f;
            kap[jp] = pk(v0 ? s0 * (float)(mu0 + nu0) : 0.f, v1 ? s1 * (float)(mu1 + nu1) : 0.f);
#pragma unroll
            for (int i = 0; i < TR; i++) {
                const double d0 = excess_at_eta(cp, cw, mu0, nu0, Lk, eta[i]);
                const double d1 = excess_at_eta(cp, cw, mu1, nu1, Lk, eta[i]);
                dd[i][jp] = pk(v0 && rvalid[i] ? s0 * (float)d0 : 0.f, v1 && rvalid[i] ? s1 * (float)d1 : 0.f);
                acc[i][jp] = 0ull;
            }
        }
        // One power of two S per warp tile with |kappa (x - eta) + W| <= S for every cell and every
        // x in [0, L].  The loop sums fma_sat(kappa / S, x - eta, W / S) = max(excess, 0) / S, and the
        // fold multiplies the reduced sums by S.  Scaling by a power of two changes no rounding, so
        // the sums equal those of a separate max per term, with the max folded into the FMA.
        double wmax = 1.0;
#pragma unroll
        for (int jp = 0; jp < TL / 2; jp++) {
            float k0, k1;
            upk(kap[jp], k0, k1);
#pragma unroll
            for (int i = 0; i < TR; i++) {
                float d0, d1;
                upk(dd[i][jp], d0, d1);
                const double xm = fmax(fabs(eta[i]), fabs(Lk - eta[i]));  // largest |x - eta|
                wmax = fmax(wmax, fmax(fabs((double)k0) * xm + fabs((double)d0), fabs((double)k1) * xm + fabs((double)d1)));
            }
        }
        int sexp;
        (void)frexp(wmax, &sexp);  // wmax < 2^sexp
        const float S = ldexpf(1.f, sexp), invS = ldexpf(1.f, -sexp);
#pragma unroll
        for (int jp = 0; jp < TL / 2; jp++) {
            float k0, k1;
            upk(kap[jp], k0, k1);
            kap[jp] = pk(k0 * invS, k1 * invS);
#pragma unroll
            for (int i = 0; i < TR; i++) {
                float d0, d1;
                upk(dd[i][jp], d0, d1);
                dd[i][jp] = pk(d0 * invS, d1 * invS);
            }
        }
        // one load: two samples' excesses for every cell of the tile.  The two samples' excesses are
        // added to each other before they join the running sum: the same number of adds, half as
        // many additions into the long sum.
        auto step = [&](const float4 v) {
#pragma unroll
            for (int i = 0; i < TR; i++) {
                // x - eta of the load's two samples in one packed add (v.x and v.z: one copy of each)
                const u64 xab = fadd2(pk(v.x, v.z), noff[i]);
                float xa0, xb0;
                upk(xab, xa0, xb0);
#pragma unroll
                for (int jp = 0; jp < TL / 2; jp++) {
                    float k0, k1, d0, d1;
                    upk(kap[jp], k0, k1);
                    upk(dd[i][jp], d0, d1);
                    const float a0 = fma_sat(k0, xa0, d0), a1 = fma_sat(k1, xa0, d1);
                    const float b0 = fma_sat(k0, xb0, d0), b1 = fma_sat(k1, xb0, d1);
                    acc[i][jp] = fadd2(acc[i][jp], fadd2(pk(a0, a1), pk(b0, b1)));
                }
            }
        };
        for (int c = 0; c < nchunks; c++) {
            const int s = c % C::STAGES;
            if (!mbar_wait_bounded(smem_u32(&full[s]), (uint32_t)((c / C::STAGES) & 1), a.wait_ns)) timeout = true;
            if (!timeout) {
                const int cnt = (int)min((int64_t)C::CHUNK, np - (int64_t)c * C::CHUNK);
                const float4* q = reinterpret_cast<const float4*>(ring + (size_t)s * C::CHUNK);
                const int nq = cnt >> 6;  // float4 (two samples) per lane: (x', x') pairs
                if (nq == C::CHUNK / 64) {  // a full chunk: a fixed trip count, unrolled with no remainder
#pragma unroll(C::UNROLL)
                    for (int t = 0; t < C::CHUNK / 64; t++) step(q[lane + 32 * t]);
                } else {
#pragma unroll 1
                    for (int t = 0; t < nq; t++) step(q[lane + 32 * t]);
                }
                // Every C::FLUSH chunks (and after the last), fold the FP32 partials into the FP64
                // accumulator of the lane's cell.
                if ((c + 1) % C::FLUSH == 0 || c + 1 == nchunks) {
                    float vals[V];
#pragma unroll
                    for (int i = 0; i < TR; i++)
#pragma unroll
                        for (int jp = 0; jp < TL / 2; jp++) {
                            upk(acc[i][jp], vals[i * TL + 2 * jp], vals[i * TL + 2 * jp + 1]);
                            acc[i][jp] = 0ull;
                        }
                    acc64 += (double)transpose_reduce<float, V>(vals, lane) * (double)S;
                }
            }
            consumed = c;
            if (__syncthreads_or(timeout)) {
                timeout = true;
                break;
            }
            if (c + C::STAGES < nchunks) {
                if (tid == 0) {
                    fence_proxy_async();
                    issue(c + C::STAGES);
                }
                issued = c + C::STAGES + 1;
            }
        }
    } else if constexpr (P == Prec::F64) {
        // each row's excess about its reservation, as in the FP32 kernel: x - eta per sample and row
        const double offd = (double)stage_offset(a.L[k]);  // the staged samples carry the class's offset
        double base[TR];
#pragma unroll
        for (int i = 0; i < TR; i++) base[i] = offd + eta[i];  // an exact integer
        double kap[TL], dd[TR][TL], acc[TR][TL];
#pragma unroll
        for (int j = 0; j < TL; j++) {
            const int lj = lt * TL + j;
            const double l = s_lam[lj];
            const bool v = lj < a.NL;
            const double mu = fmin(l, cp), nu = fmin(l, cw);
            const double sg = use_u_split(mu, nu) ? -1.0 : 1.0;  // the split of phi this column sums
            kap[j] = v ? sg * (mu + nu) : 0.0;
#pragma unroll
            for (int i = 0; i < TR; i++) {
                dd[i][j] = (v && rvalid[i]) ? sg * excess_at_eta(cp, cw, mu, nu, Lk, eta[i]) : 0.0;
                acc[i][j] = 0.0;
            }
        }
        for (int c = 0; c < nchunks; c++) {
            const int s = c % C::STAGES;
            if (!mbar_wait_bounded(smem_u32(&full[s]), (uint32_t)((c / C::STAGES) & 1), a.wait_ns)) timeout = true;
            if (!timeout) {
                const int cnt = (int)min((int64_t)C::CHUNK, np - (int64_t)c * C::CHUNK);
                const float4* q = reinterpret_cast<const float4*>(ring + (size_t)s * C::CHUNK);
                const int nq = cnt >> 6;
                for (int t = 0; t < nq; t++) {
                    const float4 v = q[lane + 32 * t];
#pragma unroll
                    for (int i = 0; i < TR; i++) {
                        const double xa = (double)v.x - base[i], xb = (double)v.z - base[i];  // x - eta, exact
#pragma unroll
                        for (int j = 0; j < TL; j++) {
                            acc[i][j] += relu(fma(kap[j], xa, dd[i][j]));
                            acc[i][j] += relu(fma(kap[j], xb, dd[i][j]));
                        }
                    }
                }
            }
            consumed = c;
            if (__syncthreads_or(timeout)) {
                timeout = true;
                break;
            }
            if (c + C::STAGES < nchunks) {
                if (tid == 0) {
                    fence_proxy_async();
                    issue(c + C::STAGES);
                }
                issued = c + C::STAGES + 1;
            }
        }
        if (!timeout) {
            double vals[V];
#pragma unroll
            for (int i = 0; i < TR; i++)
#pragma unroll
                for (int j = 0; j < TL; j++) vals[i * TL + j] = acc[i][j];
            acc64 = transpose_reduce<double, V>(vals, lane);
        }
    } else {
        // EXACT: per cell (i, j) the active samples are x >= t_ij for an integer threshold t_ij, and
        // sum_n max(kappa x_n + d, 0) = kappa sum_{x >= t} x + d #{x >= t}.  With c = t - 1,
        // max(x - c, 0) = (x - c + |x - c|) / 2 and sum_n (x - c) has a closed form, so the kernel
        // streams sum_n |x - c| only, on two pipes at once.  For half of a warp's lam columns one
        // packed FP32 add forms y = x' + (1 - t - 2^23) = x - c for two cells and one adds |y| into
        // the running sum (the absolute value rides on the add's operand); for the other half one
        // integer absolute-difference-and-add (__sad) works on the staged float's bit pattern,
        // 0x4B000000 + x.  Every value is an integer below 2^24, so both are exact.  Sums are
        // folded into int64 through the warp transposition before an FP32 sum could pass 2^24.  The
        // count #{x >= t} comes from the class's cumulative counts; the epilogue puts every sample
        // on its branch of phi with these integer sums (branch_sum) in FP64.
        constexpr int TLF = C::FCOLS;  // lam columns per r row on the packed FP32 adds (in pairs)
        constexpr int TLI = TL - TLF;  // lam columns per r row on the integer path
        static_assert(TLF % 2 == 0 && TLI >= 1, "packed columns come in pairs");
        constexpr int NPF = TLF > 0 ? TLF / 2 : 1;  // array extent (unused when TLF = 0)
        u64 ntf[TR][NPF], accf[TR][NPF];           // ntf: 1 - t - 2^23 for a pair of cells
        int cci[TR][TLI];                          // 0x4B000000 + t - 1 per cell
        unsigned acci[TR][TLI];
        // Each lane works out the threshold of the cell it owns after the final transposition
        // (cell lane >> (5 - LOG2V)); the warp's V thresholds then reach every lane by shuffles.
        const int cidx = lane >> (5 - LOG2V);
        const int ci = cidx / TL, cj = cidx % TL;
        const int c_ri = r_cta0 + r_local0 + ci, c_lj = lt * TL + cj;
        const bool c_valid = c_ri < a.R && c_lj < a.NL;
        const double c_lam = s_lam[c_lj];  // s_lam is padded with zeros to NLpad
        const double c_mu = fmin(c_lam, cp), c_kap = c_mu + fmin(c_lam, cw);
        const double c_eta = c_valid ? (double)a.r[c_ri] - (double)a.L_in[k] : 0.0;
        const double c_d = excess_offset(cp, cw, c_mu, Lk, c_eta);
        // t = L + 1 means "none" (no sample exceeds L); t in [0, L + 1] keeps |x - c| <= L + 1
        const int c_t = (int)(c_valid ? first_active(c_kap, c_d, a.L[k]) : (int64_t)a.L[k] + 1);
#pragma unroll
        for (int i = 0; i < TR; i++) {
#pragma unroll
            for (int jp = 0; jp < TLF / 2; jp++) {
                const int t0 = __shfl_sync(0xffffffffu, c_t, (i * TL + 2 * jp) << (5 - LOG2V));
                const int t1 = __shfl_sync(0xffffffffu, c_t, (i * TL + 2 * jp + 1) << (5 - LOG2V));
                ntf[i][jp] = pk((float)(1 - t0 - (1 << 23)), (float)(1 - t1 - (1 << 23)));  // exact: below 2^24
                accf[i][jp] = 0ull;
            }
#pragma unroll
            for (int jj = 0; jj < TLI; jj++) {
                cci[i][jj] = kStageBits - 1 + __shfl_sync(0xffffffffu, c_t, (i * TL + TLF + jj) << (5 - LOG2V));
                acci[i][jj] = 0u;
            }
        }
        // Fold after `fe` loads of two samples, when a lane's sums are at most 2 fe (L + 1): with
        // packed columns that is at most 2^24 (exact in FP32; the transposition's 32-lane sums stay
        // below 2^29); with none, only the integer limit applies (32 lanes' sums below 2^32).  fe
        // is a power of two, the same for every thread of the CTA.
        const int64_t fold_lim = TLF > 0 ? (1ll << 24) : (1ll << 32) / 32 - 1;
        int fe = 1;
        while (fe < (1 << 20) && 2ll * (2 * fe) * ((int64_t)a.L[k] + 1) <= fold_lim) fe <<= 1;
        long long acc_r = 0;
        auto fold = [&]() {
            unsigned vs[V];
#pragma unroll
            for (int i = 0; i < TR; i++) {
#pragma unroll
                for (int jp = 0; jp < TLF / 2; jp++) {
                    float a0, a1;
                    upk(accf[i][jp], a0, a1);
                    vs[i * TL + 2 * jp] = __float2uint_rn(a0);
                    vs[i * TL + 2 * jp + 1] = __float2uint_rn(a1);
                    accf[i][jp] = 0ull;
                }
#pragma unroll
                for (int jj = 0; jj < TLI; jj++) {
                    vs[i * TL + TLF + jj] = acci[i][jj];
                    acci[i][jj] = 0u;
                }
            }
            acc_r += (long long)transpose_reduce<unsigned, V>(vs, lane);
        };
        // one load: two samples' (x', x') pairs into every cell's sum (the compiler interleaves the
        // two pipes' instructions)
        auto step = [&](const float4 v) {
            const u64 xa = pk(v.x, v.y), xb = pk(v.z, v.w);
            const int ba = __float_as_int(v.x), bb = __float_as_int(v.z);  // 0x4B000000 + x
#pragma unroll
            for (int i = 0; i < TR; i++) {
#pragma unroll
                for (int p = 0; p < TLF / 2; p++)
                    accf[i][p] = fadd2(accf[i][p], fadd2(abs2(fadd2(xa, ntf[i][p])), abs2(fadd2(xb, ntf[i][p]))));
#pragma unroll
                for (int jj = 0; jj < TLI; jj++) acci[i][jj] = __sad(bb, cci[i][jj], __sad(ba, cci[i][jj], acci[i][jj]));
            }
        };
        auto run = [&](const float4* q, int t0, int t1, bool clamp) {
            if (clamp) {
#pragma unroll 1
                for (int t = t0; t < t1; t++) {
                    float4 v = q[lane + 32 * t];  // NaN padding -> x = 0 (x' = 2^23)
                    v.x = fmaxf(v.x, kStageOffset), v.y = fmaxf(v.y, kStageOffset);
                    v.z = fmaxf(v.z, kStageOffset), v.w = fmaxf(v.w, kStageOffset);
                    step(v);
                }
            } else {
#pragma unroll(C::UNROLL)
                for (int t = t0; t < t1; t++) step(q[lane + 32 * t]);
            }
        };
        constexpr int kChunkLoads = C::CHUNK / 64;  // loads of one full chunk per lane
        constexpr int kSegLoads = 32;
        static_assert(kChunkLoads % kSegLoads == 0, "a full chunk splits into whole segments");
        const int64_t n_k = a.N[k];
        int pending = 0;  // loads since the last fold
        for (int c = 0; c < nchunks; c++) {
            const int s = c % C::STAGES;
            if (!mbar_wait_bounded(smem_u32(&full[s]), (uint32_t)((c / C::STAGES) & 1), a.wait_ns)) timeout = true;
            if (!timeout) {
                const int cnt = (int)min((int64_t)C::CHUNK, np - (int64_t)c * C::CHUNK);
                const float4* q = reinterpret_cast<const float4*>(ring + (size_t)s * C::CHUNK);
                const int nq = cnt >> 6;
                // loads [0, t_clean) hold samples only; the class's last ones may hold NaN padding,
                // which they read as x = 0 (x' = 2^23)
                const int64_t left = n_k - (int64_t)c * C::CHUNK;
                const int t_clean = left <= 0 ? 0 : (int)min((int64_t)nq, left >> 6);
                if (nq == kChunkLoads && t_clean == nq && fe >= kSegLoads) {
                    // a full chunk of samples only: segments of a fixed trip count, which unroll with
                    // no remainder.  fe is a power of two >= kSegLoads and every earlier chunk took
                    // this path too (only a class's last chunk is ragged or padded), so the loads
                    // since the last fold are a multiple of kSegLoads and reach fe exactly at a
                    // segment's end.
#pragma unroll 1
                    for (int h = 0; h < kChunkLoads / kSegLoads; h++) {
#pragma unroll(C::UNROLL)
                        for (int t = 0; t < kSegLoads; t++) step(q[lane + 32 * (kSegLoads * h + t)]);
                        pending += kSegLoads;
                        if (pending >= fe) {
                            fold();
                            pending = 0;
                        }
                    }
                } else {
                    for (int t0 = 0; t0 < nq; t0 += fe) {
                        const int t1 = min(nq, t0 + fe);
                        const int tm = max(t0, min(t1, t_clean));
                        if (pending + (t1 - t0) > fe) {  // fold first: the loads since the last fold would pass fe
                            fold();
                            pending = 0;
                        }
                        run(q, t0, tm, false);
                        if (tm < t1) run(q, tm, t1, true);
                        pending += t1 - t0;
                        if (pending >= fe) {
                            fold();
                            pending = 0;
                        }
                    }
                }
            }
            consumed = c;
            if (__syncthreads_or(timeout)) {
                timeout = true;
                break;
            }
            if (c + C::STAGES < nchunks) {
                if (tid == 0) {
                    fence_proxy_async();
                    issue(c + C::STAGES);
                }
                issued = c + C::STAGES + 1;
            }
        }
        if (!timeout) {
            if (pending > 0) fold();
            // this lane's cell: the active count from the cumulative counts, then the branch sums
            const long long t = (long long)c_t;  // integer in [0, L + 1]
            const long long Nk = a.N[k];
            const long long count = t <= 0 ? Nk : (t > a.L[k] ? 0 : Nk - (long long)a.cdf[a.hist_off[k] + t - 1]);
            // acc_r = sum |x - c| over the samples and the padding zeros; with y = x - c,
            // max(y, 0) = (y + |y|) / 2
            const long long npad = np - Nk;
            const long long sum_abs = acc_r - npad * (t > 1 ? t - 1 : 1 - t);
            const long long sum_y = a.sumx[k] + Nk * (1 - t);
            const long long sum_relu = (sum_y + sum_abs) / 2;  // each sample adds y + |y| = 2 relu(y)
            const long long sum = sum_relu + (t - 1) * count;  // sum_{x >= t} x
            // each sample on its own branch of phi (exact integer sums): V = c_w eta - nu x below t,
            // U = c_p (L - eta) - mu (L - x) from t on; no large term cancels another
            acc64 = branch_sum(cp, cw, c_mu, fmin(c_lam, cw), Lk, c_eta, (double)Nk, count, a.sumx[k] - sum,
                               (long long)a.L[k] * count - sum);
        }
    }

    if (timeout) {
        // Report, then let every copy this CTA issued land before the CTA's shared memory is released.
        if (tid == 0) {
            atomicOr(a.err + 1, kErrTimeout);
            for (int c = consumed; c < issued; c++)
                (void)mbar_wait_bounded(smem_u32(&full[c % C::STAGES]), (uint32_t)((c / C::STAGES) & 1), a.wait_ns);
        }
        __syncthreads();
        return;
    }

    // S for this lane's cell.
    {
        const int cidx = lane >> (5 - LOG2V);
        const int i = cidx / TL, j = cidx % TL;
        const int ri = r_cta0 + r_local0 + i, lj = lt * TL + j;
        const bool owner = (lane & ((1 << (5 - LOG2V)) - 1)) == 0;
        if (owner && ri < a.R && lj < a.NL) {
            const double mu = fmin(s_lam[lj], cp), nu = fmin(s_lam[lj], cw);
            const double Nk = (double)a.N[k];
            const double eta_i = (double)a.r[ri] - (double)a.L_in[k];
            double tot;
            if constexpr (P == Prec::EXACT) {
                tot = acc64;  // the branch sums, formed above
            } else {
                // the split's base plus its excess sum: sum V + sum max(kappa x + d, 0), or
                // sum U + sum max(-(kappa x + d), 0)
                const long long N64 = a.N[k], sx = a.sumx[k];
                const double base = use_u_split(mu, nu)
                                        ? cp * (Lk - eta_i) * Nk - mu * (double)((long long)a.L[k] * N64 - sx)
                                        : cw * eta_i * Nk - nu * (double)sx;
                tot = base + acc64;
            }
            const double S = tot * s_inv_n;
            s_S[(r_local0 + i) * NLpad + lj] = S;
            if (a.S_out) {
                const size_t o = (((size_t)m * a.K + k) * a.R + ri) * a.NL_out + a.lam0 + lj;
                if (P == Prec::F32 || a.f32_out) static_cast<float*>(a.S_out)[o] = (float)S;
                else static_cast<double*>(a.S_out)[o] = S;
            }
        }
    }
    __syncthreads();

    if (P == Prec::F32 || a.f32_out) cta_epilogue<true>(a, s_S, s_lam, s_eps, NLpad, a.RG * TR, r_cta0, m, k);
    else cta_epilogue<false>(a, s_S, s_lam, s_eps, NLpad, a.RG * TR, r_cta0, m, k);
}

// The same cells in O(1) each from the class's cumulative counts C[v] = #{x <= v} and sums
// CS[v] = sum_{x <= v} x: the samples with kappa x + d > 0 are exactly x >= t for the integer
// threshold t, so sum_n max(kappa x_n + d, 0) = kappa (sum - CS[t-1]) + d (N - C[t-1]).
constexpr int kEnvR = 8;          // r values per CTA
constexpr int kEnvThreads = 256;
constexpr int kEnvTable = 4096;   // lam * eps products kept in shared memory when NL * E is at most this

// Order key of a double for the minimum over lam: equal for equal values (-0 is taken as +0) and
// ordered as the values are for every non-NaN double, so the comparison runs on integers instead
// of the FP64 pipe (which this part executes at 2 operations per clock per SM).
__device__ __forceinline__ long long order_key(double v) {
    long long b = __double_as_longlong(v);
    if (b == (long long)0x8000000000000000ull) b = 0;
    return b ^ ((b >> 63) & 0x7fffffffffffffffll);
}

// The envelope kernel's epilogue: each thread takes whole (r, eps) pairs and scans lam in
// ascending order with a strict comparison, so ties keep the lowest index (as cta_epilogue's
// reduction does); the cost of every lam is lam * eps + S, rounded as there.  One FP64 add per
// (r, eps, lam) when the CTA holds the lam * eps products (s_le, [lam][eps]), else a multiply and
// an add; no shuffles.
__device__ __forceinline__ void env_epilogue(const GridArgs& a, const double* s_S, const double* s_lam,
                                             const double* s_eps, const double* s_le, int r_cta0, int m, int k) {
    for (int p = threadIdx.x; p < kEnvR * a.E; p += blockDim.x) {
        const int rl = p / a.E, e = p % a.E;
        const int ri = r_cta0 + rl;
        if (ri >= a.R) continue;
        const double eps = s_eps[e];
        const double* S = s_S + rl * a.NL;
        double best = __dadd_rn(s_le ? s_le[e] : __dmul_rn(s_lam[0], eps), S[0]);
        long long best_key = order_key(best);
        int bj = 0;
        if (s_le) {
            for (int j = 1; j < a.NL; j++) {
                const double v = __dadd_rn(s_le[j * a.E + e], S[j]);
                const long long key = order_key(v);
                if (key < best_key) {
                    best_key = key;
                    best = v;
                    bj = j;
                }
            }
        } else {
            for (int j = 1; j < a.NL; j++) {
                const double v = __dadd_rn(__dmul_rn(s_lam[j], eps), S[j]);
                const long long key = order_key(v);
                if (key < best_key) {
                    best_key = key;
                    best = v;
                    bj = j;
                }
            }
        }
        const size_t row = ((size_t)m * a.E + e) * a.K + k;
        const size_t o = row * a.R + ri;
        static_cast<double*>(a.cost_out)[o] = best;
        if (a.lam_idx_out) a.lam_idx_out[o] = bj + a.lam0;
        const u64 key = ((u64)__double_as_longlong(best > 0.0 ? best : 0.0) & ~0xFFFFFull) | (u64)ri;
        atomicMin(a.keys + row, key);
    }
}

__global__ void __launch_bounds__(kEnvThreads) k_envelope(const GridArgs a) {
    extern __shared__ __align__(16) double esm[];
    double* s_lam = esm;
    double* s_eps = s_lam + a.NL;
    double* s_S = s_eps + a.E;
    int b = blockIdx.x;
    const int rb = b % a.r_blocks;
    b /= a.r_blocks;
    const int k = b % a.K;
    const int m = a.m0 + b / a.K;
    const int r_cta0 = rb * kEnvR;
    for (int i = threadIdx.x; i < a.NL; i += blockDim.x) s_lam[i] = a.lam[i];
    for (int i = threadIdx.x; i < a.E; i += blockDim.x) s_eps[i] = a.eps[i];
    __syncthreads();
    double* s_le = a.NL * a.E <= kEnvTable ? s_S + kEnvR * a.NL : nullptr;  // [lam][eps] products
    if (s_le)
        for (int i = threadIdx.x; i < a.NL * a.E; i += blockDim.x) s_le[i] = __dmul_rn(s_lam[i / a.E], s_eps[i % a.E]);
    const double cp = a.cp[m], cw = a.cw[m];
    const int32_t Lk = a.L[k];
    const int64_t Nk = a.N[k];
    const double N = (double)Nk, inv_n = 1.0 / N;
    const int32_t* C = a.cdf + a.hist_off[k];
    const int64_t* CS = a.csum + a.hist_off[k];
    for (int cell = threadIdx.x; cell < kEnvR * a.NL; cell += blockDim.x) {
        const int rl = cell / a.NL, j = cell % a.NL;
        const int ri = r_cta0 + rl;
        if (ri >= a.R) continue;
        const double eta = (double)a.r[ri] - (double)a.L_in[k];
        const double lam = s_lam[j];
        const double mu = fmin(lam, cp), nu = fmin(lam, cw), kap = mu + nu;
        const double d = excess_offset(cp, cw, mu, (double)Lk, eta);
        const int64_t t = first_active(kap, d, Lk);  // first active sample value, in [0, L + 1]
        const int64_t below_n = t >= 1 ? (int64_t)C[t - 1] : 0;
        const int64_t below_s = t >= 1 ? CS[t - 1] : 0;
        const int64_t cnt = Nk - below_n, sx = a.sumx[k] - below_s;  // samples from t on, and their sum
        const double tot = branch_sum(cp, cw, mu, nu, (double)Lk, eta, N, cnt, below_s, (int64_t)Lk * cnt - sx);
        const double S = tot * inv_n;
        s_S[rl * a.NL + j] = S;
        if (a.S_out) static_cast<double*>(a.S_out)[(((size_t)m * a.K + k) * a.R + ri) * a.NL_out + a.lam0 + j] = S;
    }
    __syncthreads();
    env_epilogue(a, s_S, s_lam, s_eps, s_le, r_cta0, m, k);
}

template <Prec P>
__global__ void k_finalize(const FinalizeArgs a) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)a.M * a.E * a.K) return;
    const int k = (int)(i % a.K);
    const u64 key = a.keys[i];
    if (key == ~0ull) {  // no r evaluated (cannot happen for R >= 1); report an invalid index
        if (a.r_idx) a.r_idx[i] = -1;
        return;
    }
    const int ri = (int)(P == Prec::F32 ? (key & 0xffffffffull) : (key & 0xFFFFFull));
    if (a.r_idx) a.r_idx[i] = ri;
    if (a.min_cost) {
        if constexpr (P == Prec::F32)
            static_cast<float*>(a.min_cost)[i] = __uint_as_float((uint32_t)(key >> 32));
        else
            static_cast<double*>(a.min_cost)[i] = static_cast<const double*>(a.cost)[i * a.R + ri];
    }
    if (a.fhat) {
        const int32_t v = a.r[ri] - a.L_in[k];
        a.fhat[i] = (double)a.cdf[a.hist_off[k] + v] / (double)a.N[k];
    }
}

}  // namespace

template <class C>
GridShape shape_for(int variant, int32_t R, int32_t NL, int32_t E) {
    GridShape sh;
    sh.variant = variant;
    sh.LT = (NL + C::TL - 1) / C::TL;
    sh.RG = sh.LT >= kWarpsTarget ? 1 : kWarpsTarget / sh.LT;
    sh.threads = 32 * sh.LT * sh.RG;
    sh.r_blocks = (R + sh.RG * C::TR - 1) / (sh.RG * C::TR);
    sh.smem = smem_layout(sh.RG, C::TR, sh.LT * C::TL, E, C::CHUNK, C::STAGES).total;
    return sh;
}

GridShape grid_shape(Prec p, int32_t R, int32_t NL, int32_t E, int32_t max_L) {
    if (p == Prec::ENVELOPE) {
        GridShape sh;
        sh.variant = 4;
        sh.LT = 1;
        sh.RG = 1;
        sh.threads = kEnvThreads;
        sh.r_blocks = (R + kEnvR - 1) / kEnvR;
        sh.smem = 8 * ((size_t)NL + E + (size_t)kEnvR * NL + ((int64_t)NL * E <= kEnvTable ? (size_t)NL * E : 0));
        return sh;
    }
    if (p == Prec::F64) return shape_for<CfgF64>(2, R, NL, E);
    if (p == Prec::EXACT) {  // NL <= kExactLamBlock: larger grids launch in blocks
        if (NL <= kFewLam) return shape_for<CfgExactFewLam>(8, R, NL, E);
        if (max_L > kExactIntAboveL) return shape_for<CfgExactInt>(6, R, NL, E);
        return shape_for<CfgExact>(3, R, NL, E);
    }
    if (NL <= kWarpsTarget * CfgF32::TL) return shape_for<CfgF32>(0, R, NL, E);
    return shape_for<CfgF32Wide>(1, R, NL, E);
}

cudaError_t grid_prepare(Prec p) {
    // the largest layout any variant can need: 16 warps, 256 lam, 64 eps
    const int mx = (int)(smem_layout(16, 2, 256, 64, 4096, 4).total + 4096);
    if (p == Prec::F64) return cudaFuncSetAttribute(k_grid<CfgF64>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
    if (p == Prec::EXACT) {
        cudaError_t e = cudaFuncSetAttribute(k_grid<CfgExact>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
        if (e == cudaSuccess) e = cudaFuncSetAttribute(k_grid<CfgExactInt>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(k_grid<CfgExactFewLam>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
        return e;
    }
    if (p == Prec::ENVELOPE)
        return cudaFuncSetAttribute(k_envelope, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)(8 * (256 + 64 + (size_t)kEnvR * 256 + kEnvTable)));
    cudaError_t e = cudaFuncSetAttribute(k_grid<CfgF32>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(k_grid<CfgF32Wide>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
}

cudaError_t launch_grid(Prec p, const GridShape& sh, GridArgs a, cudaStream_t s) {
    a.LT = sh.LT;
    a.RG = sh.RG;
    a.r_blocks = sh.r_blocks;
    const int64_t nblocks = (int64_t)a.m_count * a.K * a.r_blocks;
    if (nblocks <= 0 || nblocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    if (p == Prec::ENVELOPE) k_envelope<<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else if (p == Prec::F64) k_grid<CfgF64><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else if (p == Prec::EXACT && sh.variant == 3) k_grid<CfgExact><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else if (p == Prec::EXACT && sh.variant == 8) k_grid<CfgExactFewLam><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else if (p == Prec::EXACT) k_grid<CfgExactInt><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else if (sh.variant == 0) k_grid<CfgF32><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    else k_grid<CfgF32Wide><<<(unsigned)nblocks, sh.threads, sh.smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_finalize(Prec p, const FinalizeArgs& a, cudaStream_t s) {
    const int64_t n = (int64_t)a.M * a.E * a.K;
    const int threads = 256;
    const unsigned blocks = (unsigned)((n + threads - 1) / threads);
    if (p == Prec::F32) k_finalize<Prec::F32><<<blocks, threads, 0, s>>>(a);
    else k_finalize<Prec::F64><<<blocks, threads, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace kvdro
