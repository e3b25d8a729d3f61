// Segmented counting sort of bounded integer samples, per-class cumulative counts, and the
// quantile gather.  The samples are their own sort keys and are bounded by L_k, so class k's
// sorted order is fully determined by its histogram over [0, L_k]: histogram -> inclusive scan
// (the cumulative count C[v] = #{x <= v}, i.e. N times the empirical CDF) -> expansion of every
// output position p into the smallest v with C[v] > p.  The expansion also writes the (x, x)
// float pairs that the grid kernel streams, NaN-padded to a multiple of kPadSamples per class.
#include <math.h>

#include "kvdro_internal.cuh"

namespace kvdro {
namespace {

constexpr int kHistThreads = 512;
constexpr int64_t kHistSlice = 1 << 16;  // samples per histogram block
constexpr int kHistSmemBins = 16384;     // bins [0, 16384) privatised in shared memory (64 KB)
constexpr int kScanThreads = 1024;
constexpr int kExpandThreads = 512;
constexpr int kExpandPerThread = 8;
constexpr int64_t kExpandTile = (int64_t)kExpandThreads * kExpandPerThread;

__device__ __forceinline__ int find_segment(const int32_t* prefix, int K, int b) {
    // largest k with prefix[k] <= b; prefix is strictly increasing, prefix[0] = 0
    int lo = 0, hi = K;
    while (hi - lo > 1) {
        int mid = (lo + hi) >> 1;
        if (prefix[mid] <= b) lo = mid; else hi = mid;
    }
    return lo;
}

__global__ void __launch_bounds__(kHistThreads) k_histogram(SortArgs a) {
    extern __shared__ int32_t sh_bins[];
    __shared__ int32_t sh_bad[kHistThreads / 32];
    __shared__ unsigned long long sh_sum[kHistThreads / 32];
    const int k = find_segment(a.hist_blocks, a.K, blockIdx.x);
    const int64_t slice = blockIdx.x - a.hist_blocks[k];
    const int64_t beg = a.offsets[k] + slice * kHistSlice;
    const int64_t end = min(a.offsets[k + 1], beg + kHistSlice);
    const int32_t Lk = a.L[k];
    const int nb = min(Lk + 1, kHistSmemBins);
    int32_t* gh = a.hist + a.hist_off[k];
    for (int v = threadIdx.x; v < nb; v += blockDim.x) sh_bins[v] = 0;
    __syncthreads();
    int bad = 0;
    unsigned long long sum = 0;
    for (int64_t i = beg + threadIdx.x; i < end; i += blockDim.x) {
        const int32_t x = __ldg(a.lengths + i);
        if (x < 0 || x > Lk) { bad++; continue; }
        sum += (unsigned long long)x;
        if (x < nb) atomicAdd(&sh_bins[x], 1);
        else atomicAdd(&gh[x], 1);
    }
    __syncthreads();
    for (int v = threadIdx.x; v < nb; v += blockDim.x) {
        const int c = sh_bins[v];
        if (c) atomicAdd(&gh[v], c);
    }
    for (int o = 16; o; o >>= 1) {
        bad += __shfl_xor_sync(0xffffffffu, bad, o);
        sum += __shfl_xor_sync(0xffffffffu, sum, o);
    }
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) { sh_bad[w] = bad; sh_sum[w] = sum; }
    __syncthreads();
    if (threadIdx.x == 0) {
        int tb = 0;
        unsigned long long ts = 0;
        for (int i = 0; i < (int)(blockDim.x >> 5); i++) { tb += sh_bad[i]; ts += sh_sum[i]; }
        if (tb) atomicAdd(a.err, tb);
        atomicAdd(reinterpret_cast<unsigned long long*>(a.sumx + k), ts);
    }
}

// Block-wide inclusive scan of one value per thread; returns the thread's inclusive prefix and
// leaves the block total in *total (all threads).
template <typename T>
__device__ __forceinline__ T block_inclusive_scan(T t, T* warp_tot, T* total) {
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    T incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const T y = __shfl_up_sync(0xffffffffu, incl, o);
        if (l >= o) incl += y;
    }
    if (l == 31) warp_tot[w] = incl;
    __syncthreads();
    if (w == 0) {
        T s = warp_tot[l];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const T y = __shfl_up_sync(0xffffffffu, s, o);
            if (l >= o) s += y;
        }
        warp_tot[l] = s;
    }
    __syncthreads();
    const T before = (w ? warp_tot[w - 1] : (T)0) + incl;
    *total = warp_tot[kScanThreads / 32 - 1];
    __syncthreads();
    return before;
}

// Per class (one block): cumulative sums sum_{x <= v} x (if requested), then the in-place
// inclusive scan of the histogram into cumulative counts.
__global__ void __launch_bounds__(kScanThreads) k_scan(SortArgs a) {
    __shared__ int32_t warp_tot[kScanThreads / 32];
    __shared__ long long warp_tot64[kScanThreads / 32];
    const int k = blockIdx.x;
    int32_t* h = a.hist + a.hist_off[k];
    const int64_t n = (int64_t)a.L[k] + 1;
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (a.csum) {
        long long* cs = reinterpret_cast<long long*>(a.csum + a.hist_off[k]);
        long long carry64 = 0;
        for (int64_t base = 0; base < n; base += (int64_t)kScanThreads * 4) {
            const int64_t i0 = base + (int64_t)threadIdx.x * 4;
            long long v[4], t = 0;
#pragma unroll
            for (int j = 0; j < 4; j++) {
                v[j] = (i0 + j < n) ? (long long)(i0 + j) * h[i0 + j] : 0;
                t += v[j];
                v[j] = t;
            }
            long long total;
            const long long incl = block_inclusive_scan<long long>(t, warp_tot64, &total);
#pragma unroll
            for (int j = 0; j < 4; j++)
                if (i0 + j < n) cs[i0 + j] = carry64 + incl - t + v[j];
            carry64 += total;
        }
    }
    int32_t carry = 0;
    for (int64_t base = 0; base < n; base += (int64_t)kScanThreads * 4) {
        const int64_t i0 = base + (int64_t)threadIdx.x * 4;
        int32_t v[4], t = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            v[j] = (i0 + j < n) ? h[i0 + j] : 0;
            t += v[j];
            v[j] = t;
        }
        int32_t incl = t;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
            if (l >= o) incl += y;
        }
        if (l == 31) warp_tot[w] = incl;
        __syncthreads();
        if (w == 0) {
            int32_t s = warp_tot[l];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(0xffffffffu, s, o);
                if (l >= o) s += y;
            }
            warp_tot[l] = s;  // inclusive prefix of warp totals
        }
        __syncthreads();
        const int32_t before = carry + (w ? warp_tot[w - 1] : 0) + incl - t;
#pragma unroll
        for (int j = 0; j < 4; j++)
            if (i0 + j < n) h[i0 + j] = before + v[j];
        carry += warp_tot[kScanThreads / 32 - 1];
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kExpandThreads) k_expand(SortArgs a) {
    const int k = find_segment(a.exp_blocks, a.K, blockIdx.x);
    const int64_t tile = blockIdx.x - a.exp_blocks[k];
    const int64_t Nk = a.offsets[k + 1] - a.offsets[k];
    const int64_t padk = a.pair_off[k + 1] - a.pair_off[k];
    const int32_t* C = a.hist + a.hist_off[k];
    const int32_t Lk = a.L[k];
    const int64_t p0 = tile * kExpandTile + (int64_t)threadIdx.x * kExpandPerThread;
    if (p0 >= padk) return;
    int32_t* out = a.sorted + a.offsets[k];
    float2* pr = a.pairs + a.pair_off[k];
    float vals[kExpandPerThread];
    if (p0 < Nk) {
        // smallest v with C[v] > p0 (C[Lk] = Nk > p0 guarantees existence)
        int32_t lo = 0, hi = Lk;
        while (lo < hi) {
            const int32_t mid = (lo + hi) >> 1;
            if ((int64_t)__ldg(C + mid) > p0) hi = mid; else lo = mid + 1;
        }
        int32_t v = lo;
#pragma unroll
        for (int j = 0; j < kExpandPerThread; j++) {
            const int64_t p = p0 + j;
            if (p < Nk) {
                if ((int64_t)__ldg(C + v) <= p) {
                    // Galloping search for the next bin: doubling steps, then bisection.  Gaps between
                    // consecutive sorted values can span thousands of empty bins in a heavy tail.
                    int32_t base = v, step = 1;  // invariant: C[base] <= p
                    while (step <= Lk - base && (int64_t)__ldg(C + base + step) <= p) {
                        base += step;
                        step <<= 1;
                    }
                    int32_t a = min(base + 1, Lk), b2 = (step <= Lk - base) ? base + step : Lk;  // both <= Lk
                    while (a < b2) {
                        const int32_t mid = (a + b2) >> 1;
                        if ((int64_t)__ldg(C + mid) > p) b2 = mid; else a = mid + 1;
                    }
                    v = a;
                }
                out[p] = v;
                vals[j] = (float)v;
            } else {
                vals[j] = __int_as_float(0x7fc00000);  // quiet NaN pad
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < kExpandPerThread; j++) vals[j] = __int_as_float(0x7fc00000);
    }
    // p0 is a multiple of 8 and the region starts on a multiple of 128 pairs: 64-byte aligned.
    float4* dst = reinterpret_cast<float4*>(pr + p0);
#pragma unroll
    for (int j = 0; j < kExpandPerThread / 2; j++) {
        const int64_t p = p0 + 2 * j;
        if (p + 1 < padk) dst[j] = make_float4(vals[2 * j], vals[2 * j], vals[2 * j + 1], vals[2 * j + 1]);
        else if (p < padk) pr[p] = make_float2(vals[2 * j], vals[2 * j]);
    }
}

__global__ void k_gather_quantiles(const int32_t* sorted, const int64_t* offsets, const int32_t* rank, int32_t K,
                                   int32_t F, int32_t* out) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (int64_t)K * F) return;
    const int k = (int)(i / F);
    out[i] = sorted[offsets[k] + rank[i] - 1];
}

}  // namespace

cudaError_t launch_histogram(const SortArgs& a, int32_t nblocks, cudaStream_t s) {
    // per-device attribute; cheap enough to set on every launch
    cudaError_t e = cudaFuncSetAttribute(k_histogram, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kHistSmemBins * (int)sizeof(int32_t));
    if (e != cudaSuccess) return e;
    k_histogram<<<nblocks, kHistThreads, kHistSmemBins * sizeof(int32_t), s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_scan(const SortArgs& a, cudaStream_t s) {
    k_scan<<<a.K, kScanThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_expand(const SortArgs& a, int32_t nblocks, cudaStream_t s) {
    k_expand<<<nblocks, kExpandThreads, 0, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_gather_quantiles(const int32_t* sorted, const int64_t* offsets, const int32_t* rank, int32_t K,
                                    int32_t F, int32_t* out, cudaStream_t s) {
    const int64_t n = (int64_t)K * F;
    const int threads = 256;
    k_gather_quantiles<<<(unsigned)((n + threads - 1) / threads), threads, 0, s>>>(sorted, offsets, rank, K, F, out);
    return cudaGetLastError();
}

int64_t hist_slice_samples() { return kHistSlice; }
int64_t expand_tile_positions() { return kExpandTile; }

}  // namespace kvdro
