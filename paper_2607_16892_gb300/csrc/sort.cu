// Segmented counting sort of bounded integer samples, per-class cumulative counts, and the
// quantile gather.  The samples are their own sort keys and are bounded by L_k, so class k's
// sorted order is fully determined by its histogram over [0, L_k]: histogram -> inclusive scan
// (the cumulative count C[v] = #{x <= v}, i.e. N times the empirical CDF) -> expansion of every
// output position p into the smallest v with C[v] > p.  The scan also records, for every tile of
// kExpandTile output positions, the bin its first position falls in; the expansion then marks
// where each bin's run of positions starts inside the tile and takes a running maximum, O(N + L)
// in all.  It also writes the (x', x') float pairs that the grid kernel streams (x' = x plus the
// class's staging offset), NaN-padded to a multiple of kPadSamples per class.
#include <math.h>

#include <algorithm>

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
// Histogram slices get at least this many samples, so that counting outweighs clearing and
// flushing the block's shared bins.
constexpr int64_t kHistMinSlice = kHistSmemBins;

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
    // the class's samples in equal slices, one per block (at most kHistSlice each)
    const int64_t nblk = a.hist_blocks[k + 1] - a.hist_blocks[k];
    const int64_t slice_len = (a.offsets[k + 1] - a.offsets[k] + nblk - 1) / nblk;
    const int64_t slice = blockIdx.x - a.hist_blocks[k];
    const int64_t beg = a.offsets[k] + slice * slice_len;
    const int64_t end = min(a.offsets[k + 1], beg + slice_len);
    const int32_t Lk = a.L[k];
    const int nb = min(Lk + 1, kHistSmemBins);
    int32_t* gh = a.hist + a.hist_off[k];
    for (int v = threadIdx.x; v < nb; v += blockDim.x) sh_bins[v] = 0;
    __syncthreads();
    // Per sample: an unsigned comparison is the whole range check (a negative x wraps above L),
    // and the two atomics are predicated, so a sample costs no branch.  A thread counts at most
    // ceil(kHistSlice / kHistThreads) = 128 samples of at most 2^24, so its sum fits 32 bits.
    int bad = 0;
    uint32_t sum32 = 0;
    auto count = [&](int32_t x) {
        const bool ok = (uint32_t)x <= (uint32_t)Lk;
        bad += ok ? 0 : 1;
        sum32 += ok ? (uint32_t)x : 0u;
        const bool in_smem = ok && x < nb, in_gmem = ok && x >= nb;
        if (in_smem) atomicAdd(&sh_bins[x], 1);
        if (in_gmem) atomicAdd(&gh[x], 1);
    };
    // 16-byte loads of four samples over the slice's aligned middle (alignment is taken from the
    // address: `lengths` is the caller's pointer): each thread loads its next two vectors before
    // it counts the current two, so four loads are in flight while the atomics run; the unaligned
    // head and the tail one sample at a time.
    const int32_t* src = a.lengths;
    const int64_t mis = (int64_t)((reinterpret_cast<uintptr_t>(src + beg) >> 2) & 3);
    const int64_t vbeg = min(end, beg + ((4 - mis) & 3));
    const int64_t nvec = (end - vbeg) >> 2;
    const int64_t vend = vbeg + 4 * nvec;
    for (int64_t i = beg + threadIdx.x; i < vbeg; i += blockDim.x) count(__ldg(src + i));
    const int4* v4 = reinterpret_cast<const int4*>(src + vbeg);
    const int64_t bd = blockDim.x;
    int64_t q = threadIdx.x;
    int4 u = make_int4(0, 0, 0, 0), w = make_int4(0, 0, 0, 0);
    bool hu = q < nvec, hw = q + bd < nvec;
    if (hu) u = __ldg(v4 + q);
    if (hw) w = __ldg(v4 + q + bd);
    while (hu) {
        const int64_t qn = q + 2 * bd;
        const bool nu = qn < nvec, nw = qn + bd < nvec;
        int4 u2 = make_int4(0, 0, 0, 0), w2 = make_int4(0, 0, 0, 0);
        if (nu) u2 = __ldg(v4 + qn);
        if (nw) w2 = __ldg(v4 + qn + bd);
        count(u.x); count(u.y); count(u.z); count(u.w);
        if (hw) {
            count(w.x); count(w.y); count(w.z); count(w.w);
        }
        u = u2;
        w = w2;
        hu = nu;
        hw = nw;
        q = qn;
    }
    for (int64_t i = vend + threadIdx.x; i < end; i += blockDim.x) count(__ldg(src + i));
    __syncthreads();
    for (int v = threadIdx.x; v < nb; v += blockDim.x) {
        const int c = sh_bins[v];
        if (c) atomicAdd(&gh[v], c);
    }
    unsigned long long sum = sum32;
    for (int o = 16; o; o >>= 1) {
        bad += __shfl_xor_sync(0xffffffffu, bad, o);
        sum += __shfl_xor_sync(0xffffffffu, sum, o);
    }
    const int wid = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) { sh_bad[wid] = bad; sh_sum[wid] = sum; }
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
    // For the expansion: tile_lo[q] = the bin holding position q * kExpandTile for each tile q of
    // the class's sorted samples, and one more entry: the bin holding the last position, N - 1.
    // Every position lies in exactly one bin's run [C[v] - h[v], C[v]), so each entry is written once.
    const int64_t Nk = a.offsets[k + 1] - a.offsets[k];
    const int64_t tiles = (Nk + kExpandTile - 1) / kExpandTile;
    int32_t* tl = a.tile_lo + a.exp_blocks[k] + k;
#pragma unroll
    for (int j = 0; j < 4; j++)
        if (i0 + j < n) {
            const int64_t hi = cc + incl - t + w[j], lo = hi - cnt[j];
            h[i0 + j] = (int32_t)hi;
            if (lo < hi) {
                for (int64_t q = (lo + kExpandTile - 1) / kExpandTile; q * kExpandTile < hi && q < tiles; q++)
                    tl[q] = (int32_t)(i0 + j);
                if (lo <= Nk - 1 && Nk - 1 < hi) tl[tiles] = (int32_t)(i0 + j);
            }
        }
}

__global__ void __launch_bounds__(kExpandThreads) k_expand(SortArgs a) {
    // One tile of kExpandTile output positions [p0, p0 + kExpandTile).  Its positions fall in the
    // bins [tile_lo[q], tile_lo[q + 1]] (recorded by the scan).  The run of bin v starts at position
    // C[v - 1]; marking each non-empty bin's run start inside the tile (and the first bin at the
    // tile's first position) and taking the running maximum gives every position its value, since
    // values ascend with position.  Stores are lane-contiguous (coalesced).
    __shared__ int32_t sv[kExpandTile];
    __shared__ int32_t s_wmax[kExpandThreads / 32];
    const int k = find_segment(a.exp_blocks, a.K, blockIdx.x);
    const int64_t q = blockIdx.x - a.exp_blocks[k];
    const int64_t Nk = a.offsets[k + 1] - a.offsets[k];
    const int64_t padk = a.pair_off[k + 1] - a.pair_off[k];
    const int32_t* C = a.hist + a.hist_off[k];
    const int32_t Lk = a.L[k];
    const int64_t p0 = q * kExpandTile;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int64_t pend = min(Nk, p0 + kExpandTile);  // sample positions of this tile
    if (p0 < Nk) {  // block-uniform
        const int32_t* tl = a.tile_lo + a.exp_blocks[k] + k;
        const int32_t v_lo = tl[q], v_hi = tl[q + 1];
        for (int i = tid; i < kExpandTile; i += kExpandThreads) sv[i] = i == 0 ? v_lo : -1;
        __syncthreads();
        // a non-empty bin after v_lo starts its run after p0 (C[v - 1] >= C[v_lo] > p0)
        for (int64_t v = (int64_t)v_lo + 1 + tid; v <= v_hi; v += kExpandThreads) {
            const int32_t start = __ldg(C + v - 1);
            if (__ldg(C + v) > start && start < pend) sv[start - p0] = (int32_t)v;
        }
        __syncthreads();
        // inclusive running maximum: kExpandPerThread consecutive entries per thread, then across
        // the lanes of the warp and across the warps
        int32_t m[kExpandPerThread], run = -1;
#pragma unroll
        for (int j = 0; j < kExpandPerThread; j++) {
            run = max(run, sv[tid * kExpandPerThread + j]);
            m[j] = run;
        }
        int32_t incl = run;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int32_t y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl = max(incl, y);
        }
        if (lane == 31) s_wmax[wid] = incl;
        __syncthreads();
        if (wid == 0) {
            int32_t x = lane < kExpandThreads / 32 ? s_wmax[lane] : -1;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int32_t y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x = max(x, y);
            }
            if (lane < kExpandThreads / 32) s_wmax[lane] = x;
        }
        __syncthreads();
        const int32_t lane_before = __shfl_up_sync(0xffffffffu, incl, 1);
        const int32_t before = max(wid > 0 ? s_wmax[wid - 1] : -1, lane > 0 ? lane_before : -1);
#pragma unroll
        for (int j = 0; j < kExpandPerThread; j++) sv[tid * kExpandPerThread + j] = max(before, m[j]);
        __syncthreads();
        int32_t* out = a.sorted + a.offsets[k];
        for (int64_t i = tid; i < pend - p0; i += kExpandThreads) out[p0 + i] = sv[i];
    }
    // the tile's (x', x') pairs, two positions per 16-byte store; NaN past the class's samples
    float2* pr = a.pairs + a.pair_off[k];
    const float nan = __int_as_float(0x7fc00000);  // quiet NaN pad
    const float off = stage_offset(Lk);              // x + 2^23 is exact for L <= 2^22
    const int64_t qend = min(padk, p0 + kExpandTile);  // padk is a multiple of 128: even
    for (int64_t i = 2 * (int64_t)tid; p0 + i < qend; i += 2 * kExpandThreads) {
        const int64_t pos = p0 + i;
        const float f0 = pos < Nk ? (float)sv[i] + off : nan;
        const float f1 = pos + 1 < Nk ? (float)sv[i + 1] + off : nan;
        if (pos + 1 < qend) *reinterpret_cast<float4*>(pr + pos) = make_float4(f0, f0, f1, f1);
        else pr[pos] = make_float2(f0, f0);
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

// Histogram blocks of each class (written as a prefix over the classes): slices of at most
// kHistSlice and at least kHistMinSlice samples, as many as fill whole waves of the device's
// resident histogram blocks -- a last wave only a little filled would leave most SMs idle.
cudaError_t hist_block_prefix(const int64_t* N, int32_t K, int32_t* prefix) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_histogram, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kHistSmemBins * (int)sizeof(int32_t));
    if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_histogram, kHistThreads,
                                                          kHistSmemBins * sizeof(int32_t));
    if (e != cudaSuccess) return e;
    const int64_t slots = std::max<int64_t>(1, (int64_t)sms * per_sm);
    int64_t total = 0, base = 0;
    for (int32_t k = 0; k < K; k++) {
        total += N[k];
        base += (N[k] + kHistSlice - 1) / kHistSlice;
    }
    const int64_t target = (base + slots - 1) / slots * slots;
    const int64_t slice = std::max<int64_t>(kHistMinSlice, (total + target - 1) / target);
    prefix[0] = 0;
    for (int32_t k = 0; k < K; k++) {
        const int64_t nb = std::max<int64_t>((N[k] + kHistSlice - 1) / kHistSlice, N[k] / slice);
        prefix[k + 1] = (int32_t)std::min<int64_t>(0x7fffffffLL, prefix[k] + std::max<int64_t>(1, nb));
    }
    return cudaSuccess;
}

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
