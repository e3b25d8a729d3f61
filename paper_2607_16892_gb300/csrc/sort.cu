// Segmented counting sort of bounded integer samples, per-class cumulative counts, and the
// quantile gather.  The samples are their own sort keys and are bounded by L_k, so class k's
// sorted order is fully determined by its histogram over [0, L_k]: histogram -> inclusive scan
// (the cumulative count C[v] = #{x <= v}, i.e. N times the empirical CDF) -> expansion of every
// output position p into the smallest v with C[v] > p.  The expansion also writes the (x', x')
// float pairs that the grid kernel streams (x' = x plus the class's staging offset), NaN-padded
// to a multiple of kPadSamples per class.
#include <math.h>

#include "kvdro_internal.cuh"

namespace kvdro {
namespace {

constexpr int kHistThreads = 512;
constexpr int64_t kHistSlice = 1 << 16;  // samples per histogram block
constexpr int kHistSmemBins = 16384;     // bins [0, 16384) privatised in shared memory (64 KB)
constexpr int kScanThreads = 1024;
constexpr int64_t kScanTile = (int64_t)kScanThreads * 4;  // bins per scan block
constexpr int kExpandThreads = 512;
constexpr int kExpandPerThread = 8;
constexpr int64_t kExpandTile = (int64_t)kExpandThreads * kExpandPerThread;
constexpr int kExpandCoarse = 2048;  // entries of the per-block coarse index of cumulative counts (8 KB)

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
    auto count = [&](int32_t x) {
        if (x < 0 || x > Lk) {
            bad++;
            return;
        }
        sum += (unsigned long long)x;
        if (x < nb) atomicAdd(&sh_bins[x], 1);
        else atomicAdd(&gh[x], 1);
    };
    // 16-byte loads of four samples over the slice's aligned middle (alignment is taken from the
    // address: `lengths` is the caller's pointer), two loads in flight per thread per step;
    // the unaligned head and the tail one sample at a time.
    const int32_t* src = a.lengths;
    const int64_t mis = (int64_t)((reinterpret_cast<uintptr_t>(src + beg) >> 2) & 3);
    const int64_t vbeg = min(end, beg + ((4 - mis) & 3));
    const int64_t nvec = (end - vbeg) >> 2;
    const int64_t vend = vbeg + 4 * nvec;
    for (int64_t i = beg + threadIdx.x; i < vbeg; i += blockDim.x) count(__ldg(src + i));
    const int4* v4 = reinterpret_cast<const int4*>(src + vbeg);
    int64_t q = threadIdx.x;
    for (; q + (int64_t)blockDim.x < nvec; q += 2 * (int64_t)blockDim.x) {
        const int4 u = __ldg(v4 + q), w = __ldg(v4 + q + blockDim.x);
        count(u.x); count(u.y); count(u.z); count(u.w);
        count(w.x); count(w.y); count(w.z); count(w.w);
    }
    if (q < nvec) {
        const int4 u = __ldg(v4 + q);
        count(u.x); count(u.y); count(u.z); count(u.w);
    }
    for (int64_t i = vend + threadIdx.x; i < end; i += blockDim.x) count(__ldg(src + i));
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

// Block-wide sum of one value per thread; every thread gets the total.
template <typename T>
__device__ __forceinline__ T block_sum(T t, T* warp_tot) {
#pragma unroll
    for (int o = 16; o; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) warp_tot[w] = t;
    __syncthreads();
    T s = l < (int)(blockDim.x >> 5) ? warp_tot[l] : (T)0;
#pragma unroll
    for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    __syncthreads();  // warp_tot is reused by the caller
    return s;
}

// The cumulative counts (and sums) of every class in two passes over tiles of kScanTile bins,
// one block per (tile, class) so that every SM takes part: first each tile's count total (and
// its sum of v h[v]), then each tile's inclusive scan, offset by the totals of the class's
// earlier tiles.  The counts are scanned in place into C[v] = #{x <= v}; the sums go to
// csum[v] = sum_{x <= v} x when it is requested.
__global__ void __launch_bounds__(kScanThreads) k_scan_totals(SortArgs a) {
    __shared__ long long warp_tot[kScanThreads / 32];
    const int k = blockIdx.y;
    const int64_t n = (int64_t)a.L[k] + 1, b0 = (int64_t)blockIdx.x * kScanTile;
    if (b0 >= n) return;  // the class has fewer tiles
    const int32_t* h = a.hist + a.hist_off[k];
    long long c = 0, v = 0;
#pragma unroll
    for (int j = 0; j < 4; j++) {
        const int64_t i = b0 + (int64_t)threadIdx.x * 4 + j;
        if (i < n) {
            const long long hi = h[i];
            c += hi;
            v += i * hi;
        }
    }
    c = block_sum<long long>(c, warp_tot);
    if (a.csum) v = block_sum<long long>(v, warp_tot);
    if (threadIdx.x == 0) {
        const int64_t o = (int64_t)k * a.scan_tiles + blockIdx.x;
        a.tile_tot[2 * o] = c;
        a.tile_tot[2 * o + 1] = v;
    }
}

__global__ void __launch_bounds__(kScanThreads) k_scan_apply(SortArgs a) {
    __shared__ long long warp_tot[kScanThreads / 32];
    __shared__ int32_t warp_tot32[kScanThreads / 32];
    const int k = blockIdx.y;
    const int64_t n = (int64_t)a.L[k] + 1, b0 = (int64_t)blockIdx.x * kScanTile;
    if (b0 >= n) return;
    int32_t* h = a.hist + a.hist_off[k];
    // carry-in: the totals of this class's earlier tiles
    long long cc = 0, cv = 0;
    for (int u = threadIdx.x; u < (int)blockIdx.x; u += blockDim.x) {
        const int64_t o = (int64_t)k * a.scan_tiles + u;
        cc += a.tile_tot[2 * o];
        cv += a.tile_tot[2 * o + 1];
    }
    cc = block_sum<long long>(cc, warp_tot);
    if (a.csum) cv = block_sum<long long>(cv, warp_tot);
    const int64_t i0 = b0 + (int64_t)threadIdx.x * 4;
    int32_t cnt[4];
#pragma unroll
    for (int j = 0; j < 4; j++) cnt[j] = (i0 + j < n) ? h[i0 + j] : 0;
    if (a.csum) {
        long long* cs = reinterpret_cast<long long*>(a.csum + a.hist_off[k]);
        long long w[4], t = 0;
#pragma unroll
        for (int j = 0; j < 4; j++) {
            t += (long long)(i0 + j) * cnt[j];
            w[j] = t;
        }
        long long total;
        const long long incl = block_inclusive_scan<long long>(t, warp_tot, &total);
#pragma unroll
        for (int j = 0; j < 4; j++)
            if (i0 + j < n) cs[i0 + j] = cv + incl - t + w[j];
    }
    int32_t w[4], t = 0;
#pragma unroll
    for (int j = 0; j < 4; j++) {
        t += cnt[j];
        w[j] = t;
    }
    int32_t total;
    const int32_t incl = block_inclusive_scan<int32_t>(t, warp_tot32, &total);
#pragma unroll
    for (int j = 0; j < 4; j++)
        if (i0 + j < n) h[i0 + j] = (int32_t)(cc + incl - t + w[j]);
}

__global__ void __launch_bounds__(kExpandThreads) k_expand(SortArgs a) {
    // A coarse index of the class's cumulative counts in shared memory: entry c is C at the end of
    // bucket c (buckets of `stride` consecutive bins).  Each thread finds its first position's
    // bucket there, then the bin inside the bucket in global memory (log2(stride) steps), and
    // walks on for its next positions.  The warp then stores its 256 values lane-contiguously
    // through shared memory (rows of 9 words: conflict-free), so every store is coalesced.
    __shared__ int32_t sK[kExpandCoarse];
    __shared__ int32_t sV[kExpandThreads / 32][32 * 9];
    const int k = find_segment(a.exp_blocks, a.K, blockIdx.x);
    const int64_t tile = blockIdx.x - a.exp_blocks[k];
    const int64_t Nk = a.offsets[k + 1] - a.offsets[k];
    const int64_t padk = a.pair_off[k + 1] - a.pair_off[k];
    const int32_t* C = a.hist + a.hist_off[k];
    const int32_t Lk = a.L[k];
    const int32_t stride = (int32_t)(((int64_t)Lk + kExpandCoarse) / kExpandCoarse);  // ceil((Lk + 1) / kExpandCoarse)
    const int32_t ncoarse = (int32_t)(((int64_t)Lk + stride) / stride);                 // ceil((Lk + 1) / stride)
    for (int c = threadIdx.x; c < ncoarse; c += blockDim.x)
        sK[c] = __ldg(C + min((int64_t)Lk, (int64_t)(c + 1) * stride - 1));
    __syncthreads();
    const int lane = threadIdx.x & 31;
    int32_t* wv = sV[threadIdx.x >> 5];
    const int64_t p0 = tile * kExpandTile + (int64_t)threadIdx.x * kExpandPerThread;
    if (p0 < Nk) {
        // smallest bucket c with sK[c] > p0 (the last bucket ends at Lk and C[Lk] = Nk > p0)
        int32_t lo = 0, hi = ncoarse - 1;
        while (lo < hi) {
            const int32_t mid = (lo + hi) >> 1;
            if ((int64_t)sK[mid] > p0) hi = mid; else lo = mid + 1;
        }
        // then the smallest v in the bucket with C[v] > p0 (C at the bucket's end is sK[lo] > p0)
        int32_t a0 = lo * stride, b0 = (int32_t)min((int64_t)Lk, (int64_t)(lo + 1) * stride - 1);
        while (a0 < b0) {
            const int32_t mid = (a0 + b0) >> 1;
            if ((int64_t)__ldg(C + mid) > p0) b0 = mid; else a0 = mid + 1;
        }
        int32_t v = a0;
#pragma unroll
        for (int j = 0; j < kExpandPerThread; j++) {
            const int64_t p = p0 + j;
            if (p < Nk && (int64_t)__ldg(C + v) <= p) {
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
            wv[lane * 9 + j] = v;  // positions past Nk are never stored as samples
        }
    }
    __syncwarp();
    // lane-contiguous stores: position idx of the warp's 256 lives at wv[(idx / 8) * 9 + idx % 8]
    const int64_t wbase = tile * kExpandTile + (int64_t)(threadIdx.x >> 5) * 32 * kExpandPerThread;
    int32_t* out = a.sorted + a.offsets[k];
    float2* pr = a.pairs + a.pair_off[k];
#pragma unroll
    for (int i = 0; i < kExpandPerThread; i++) {
        const int idx = i * 32 + lane;
        const int64_t p = wbase + idx;
        if (p < Nk) out[p] = wv[(idx >> 3) * 9 + (idx & 7)];
    }
    const float nan = __int_as_float(0x7fc00000);  // quiet NaN pad
    const float off = stage_offset(Lk);              // x + 2^23 is exact for L <= 2^22
#pragma unroll
    for (int i = 0; i < kExpandPerThread / 2; i++) {
        const int idx = (i * 32 + lane) * 2;  // even: the pair store is 16-byte aligned
        const int64_t q = wbase + idx;
        if (q < padk) {
            const float f0 = q < Nk ? (float)wv[(idx >> 3) * 9 + (idx & 7)] + off : nan;
            const float f1 = q + 1 < Nk ? (float)wv[((idx + 1) >> 3) * 9 + ((idx + 1) & 7)] + off : nan;
            if (q + 1 < padk) *reinterpret_cast<float4*>(pr + q) = make_float4(f0, f0, f1, f1);
            else pr[q] = make_float2(f0, f0);
        }
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
    const dim3 grid((unsigned)a.scan_tiles, (unsigned)a.K);
    k_scan_totals<<<grid, kScanThreads, 0, s>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_scan_apply<<<grid, kScanThreads, 0, s>>>(a);
    return cudaGetLastError();
}

int64_t scan_tile_bins() { return kScanTile; }

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
