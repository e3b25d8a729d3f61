// C ABI of the library (declared in include/kvdro.h): argument validation, buffer ownership,
// host/device pointer handling and the launch sequence of each entry point.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <initializer_list>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "kvdro.h"
#include "kvdro_internal.cuh"

namespace kvdro {
int64_t hist_slice_samples();
int64_t expand_tile_positions();
int64_t scan_tile_bins();
}  // namespace kvdro

using kvdro::Prec;

namespace {

constexpr int32_t kMaxK = 4096;
constexpr int32_t kMaxL = 1 << 24;        // samples, reservations and L_in + L stay exact in FP32
constexpr int32_t kMaxR = 1 << 20;        // the FP64 argmin key keeps the r index in 20 bits
constexpr int32_t kMaxE = 64;
constexpr int32_t kMaxM = 65536;
constexpr int32_t kMaxF = 65536;
constexpr int64_t kMaxKF = 1 << 22;
constexpr long long kTestWaitNs = 1000000;  // the wait test's bound: 1 ms
constexpr int32_t kMaxNLf32 = 256;
constexpr int64_t kPartBytes = 256LL << 20;  // cap of the running-minimum buffer of lam blocks
constexpr int32_t kMaxNLf64 = 128;
// Host outputs of a grid over several regimes return in up to this many regime blocks, each
// copied while the next evaluates.
constexpr int64_t kCopyBlocks = 16;

struct Buf {
    void* p = nullptr;
    size_t bytes = 0;
};

}  // namespace

struct kvdro_ctx {
    int device = 0;
    std::string err;
    int fail_after = -1;  // test hook: the fail_after-th allocation of this context fails
    int skip_chunk = -1;  // test hook: grid kernels never copy this chunk, so their waits run out
    int allocs = 0;
    cudaStream_t last_stream = nullptr;

    bool loaded = false;
    int32_t K = 0;
    int64_t total = 0, pair_total = 0, hist_total = 0;
    std::vector<int64_t> off, pair_off, hist_off, N;
    std::vector<int32_t> L, Lin, hist_blocks, exp_blocks;

    Buf sorted, pairs, hist, csum, sumx, meta, errs, in_stage, grid_in, keys, cost64, out_stage, ranks, scan_tot, part,
        tile_lo;
    void* pin = nullptr;  // pinned host staging
    size_t pin_bytes = 0;
    cudaEvent_t pin_free = nullptr;  // completes when the last copy out of `pin` is done
    cudaEvent_t grid_t0 = nullptr, grid_t1 = nullptr;  // around the last grid-kernel launches
    // Copies of host outputs back to the caller, overlapped with later grid launches
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t copy_ready = nullptr, copy_done = nullptr;
    bool grid_timed = false;

    // device views into `meta`
    int64_t *d_off = nullptr, *d_pair_off = nullptr, *d_hist_off = nullptr, *d_N = nullptr;
    int32_t *d_L = nullptr, *d_Lin = nullptr, *d_hist_blocks = nullptr, *d_exp_blocks = nullptr;
};

namespace {

int fail(kvdro_ctx* c, int code, const char* fmt, ...) {
    if (c) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof(buf), fmt, ap);
        va_end(ap);
        c->err = buf;
    }
    return code;
}

int cuda_fail(kvdro_ctx* c, cudaError_t e, const char* what) {
    return fail(c, KVDRO_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define KV_CUDA(call, what)                            \
    do {                                               \
        cudaError_t e_ = (call);                       \
        if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
    } while (0)

// An NVTX range around one entry point (visible in Nsight timelines; a no-op without a tool).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};

// Keeps the caller's current device and restores it on exit.
struct DeviceGuard {
    int prev = -1;
    bool ok = false;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

int ensure(kvdro_ctx* ctx, Buf& b, size_t bytes) {
    if (bytes == 0) bytes = 16;
    if (b.bytes >= bytes) return KVDRO_OK;
    if (b.p) {
        cudaFree(b.p);
        b.p = nullptr;
        b.bytes = 0;
    }
    ctx->allocs++;
    if (ctx->fail_after > 0 && ctx->allocs == ctx->fail_after)
        return fail(ctx, KVDRO_ENOMEM, "device allocation of %zu bytes failed (injected by KVDRO_TEST_FAIL_ALLOC)", bytes);
    cudaError_t e = cudaMalloc(&b.p, bytes);
    if (e != cudaSuccess) {
        cudaGetLastError();
        b.p = nullptr;
        return fail(ctx, KVDRO_ENOMEM, "cudaMalloc(%zu): %s", bytes, cudaGetErrorString(e));
    }
    b.bytes = bytes;
    return KVDRO_OK;
}

void release(Buf& b) {
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.bytes = 0;
}

// Pinned staging for small host->device uploads; waits for the previous upload first.
int pinned(kvdro_ctx* ctx, size_t bytes, void** out) {
    if (ctx->pin_free) {
        cudaError_t e = cudaEventSynchronize(ctx->pin_free);
        if (e != cudaSuccess) return cuda_fail(ctx, e, "waiting for the staging buffer");
    }
    if (ctx->pin_bytes < bytes) {
        if (ctx->pin) cudaFreeHost(ctx->pin);
        ctx->pin = nullptr;
        ctx->pin_bytes = 0;
        ctx->allocs++;
        if (ctx->fail_after > 0 && ctx->allocs == ctx->fail_after)
            return fail(ctx, KVDRO_ENOMEM, "pinned allocation failed (injected by KVDRO_TEST_FAIL_ALLOC)");
        size_t want = bytes < 4096 ? 4096 : bytes;
        cudaError_t e = cudaHostAlloc(&ctx->pin, want, cudaHostAllocDefault);
        if (e != cudaSuccess) {
            cudaGetLastError();
            ctx->pin = nullptr;
            return fail(ctx, KVDRO_ENOMEM, "cudaHostAlloc(%zu): %s", want, cudaGetErrorString(e));
        }
        ctx->pin_bytes = want;
    }
    *out = ctx->pin;
    return KVDRO_OK;
}

// Device-accessible (device or managed memory) versus host memory (pinned or pageable).
bool is_device_ptr(const void* p) {
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Reads and clears the kernels' error word; KVDRO_ETIMEOUT if a bounded wait gave up.
int check_kernel_errors(kvdro_ctx* ctx, cudaStream_t s) {
    if (!ctx->errs.p) return KVDRO_OK;
    int32_t h[2] = {0, 0};
    KV_CUDA(cudaMemcpyAsync(h, ctx->errs.p, sizeof(h), cudaMemcpyDeviceToHost, s), "reading kernel status");
    KV_CUDA(cudaStreamSynchronize(s), "reading kernel status");
    if (h[1] & kvdro::kErrTimeout) {
        KV_CUDA(cudaMemsetAsync(static_cast<int32_t*>(ctx->errs.p) + 1, 0, sizeof(int32_t), s), "clearing status");
        return fail(ctx, KVDRO_ETIMEOUT, "a grid kernel gave up waiting for a staged sample chunk");
    }
    return KVDRO_OK;
}

// Every r must lie in [L_in, L_in + L_max] of every class (the reservation domain of Sec. 2.2),
// i.e. in [max_k L_in, min_k (L_in + L_max)]: O(R + K).
int check_reservations(kvdro_ctx* ctx, int32_t R, const int32_t* r) {
    int32_t k_lo = 0, k_hi = 0;
    for (int32_t k = 1; k < ctx->K; k++) {
        if (ctx->Lin[k] > ctx->Lin[k_lo]) k_lo = k;
        if ((int64_t)ctx->Lin[k] + ctx->L[k] < (int64_t)ctx->Lin[k_hi] + ctx->L[k_hi]) k_hi = k;
    }
    const int64_t lo = ctx->Lin[k_lo], hi = (int64_t)ctx->Lin[k_hi] + ctx->L[k_hi];
    for (int32_t i = 0; i < R; i++)
        if ((int64_t)r[i] < lo || (int64_t)r[i] > hi)
            return fail(ctx, KVDRO_EINVAL, "r[%d] = %d outside [L_in, L_in + L_max] of class %d", i, r[i],
                        (int64_t)r[i] < lo ? k_lo : k_hi);
    return KVDRO_OK;
}

bool finite_nonneg(const double* v, int64_t n) {
    for (int64_t i = 0; i < n; i++)
        if (!std::isfinite(v[i]) || v[i] < 0.0) return false;
    return true;
}

}  // namespace

extern "C" {

int kvdro_create(kvdro_ctx** out, int device_ordinal) {
    if (!out) return KVDRO_EINVAL;
    *out = nullptr;
    int n = 0;
    if (cudaGetDeviceCount(&n) != cudaSuccess) {
        cudaGetLastError();
        return KVDRO_ECUDA;
    }
    if (device_ordinal < 0 || device_ordinal >= n) return KVDRO_EINVAL;
    kvdro_ctx* ctx = new (std::nothrow) kvdro_ctx();
    if (!ctx) return KVDRO_ENOMEM;
    ctx->device = device_ordinal;
    if (const char* f = std::getenv("KVDRO_TEST_FAIL_ALLOC")) ctx->fail_after = std::atoi(f);
    if (const char* f = std::getenv("KVDRO_TEST_SKIP_CHUNK")) ctx->skip_chunk = std::atoi(f);
    DeviceGuard g(device_ordinal);
    if (!g.ok || kvdro::grid_prepare(Prec::F32) != cudaSuccess || kvdro::grid_prepare(Prec::F64) != cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->pin_free, cudaEventDisableTiming) != cudaSuccess ||
        kvdro::grid_prepare(Prec::EXACT) != cudaSuccess || kvdro::grid_prepare(Prec::ENVELOPE) != cudaSuccess ||
        cudaEventCreate(&ctx->grid_t0) != cudaSuccess ||
        cudaEventCreate(&ctx->grid_t1) != cudaSuccess ||
        cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->copy_ready, cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&ctx->copy_done, cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        delete ctx;
        return KVDRO_ECUDA;
    }
    *out = ctx;
    return KVDRO_OK;
}

int kvdro_destroy(kvdro_ctx* ctx) {
    if (!ctx) return KVDRO_OK;
    DeviceGuard g(ctx->device);
    if (ctx->last_stream) cudaStreamSynchronize(ctx->last_stream);
    cudaDeviceSynchronize();
    for (Buf* b : {&ctx->sorted, &ctx->scan_tot, &ctx->pairs, &ctx->hist, &ctx->csum, &ctx->sumx, &ctx->meta, &ctx->errs, &ctx->in_stage,
                   &ctx->grid_in, &ctx->keys, &ctx->cost64, &ctx->out_stage, &ctx->ranks, &ctx->part, &ctx->tile_lo})
        release(*b);
    if (ctx->pin) cudaFreeHost(ctx->pin);
    if (ctx->pin_free) cudaEventDestroy(ctx->pin_free);
    if (ctx->grid_t0) cudaEventDestroy(ctx->grid_t0);
    if (ctx->grid_t1) cudaEventDestroy(ctx->grid_t1);
    if (ctx->copy_ready) cudaEventDestroy(ctx->copy_ready);
    if (ctx->copy_done) cudaEventDestroy(ctx->copy_done);
    if (ctx->copy_stream) cudaStreamDestroy(ctx->copy_stream);
    cudaGetLastError();
    delete ctx;
    return KVDRO_OK;
}

const char* kvdro_last_error(const kvdro_ctx* ctx) { return ctx ? ctx->err.c_str() : "null context"; }

int kvdro_load_samples(kvdro_ctx* ctx, int32_t K, const int64_t* offsets, const int32_t* lengths,
                       const int32_t* L_max, const int32_t* L_in, void* stream) {
    NvtxRange nvtx_("kvdro_load_samples");
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    if (K < 1 || K > kMaxK) return fail(ctx, KVDRO_EINVAL, "K = %d outside [1, %d]", K, kMaxK);
    if (!offsets || !lengths || !L_max) return fail(ctx, KVDRO_EINVAL, "offsets, lengths and L_max are required");
    if (offsets[0] != 0) return fail(ctx, KVDRO_EINVAL, "offsets[0] must be 0");
    for (int32_t k = 0; k < K; k++) {
        const int64_t n = offsets[k + 1] - offsets[k];
        if (n < 1) return fail(ctx, KVDRO_EINVAL, "class %d has %lld samples (need >= 1)", k, (long long)n);
        if (n > 0x7fffffffLL) return fail(ctx, KVDRO_EINVAL, "class %d has more than 2^31-1 samples", k);
        if (L_max[k] < 1 || L_max[k] > kMaxL) return fail(ctx, KVDRO_EINVAL, "L_max[%d] = %d outside [1, 2^24]", k, L_max[k]);
        const int64_t lin = L_in ? L_in[k] : 0;
        if (lin < 0 || lin + L_max[k] > kMaxL) return fail(ctx, KVDRO_EINVAL, "L_in[%d] = %lld invalid", k, (long long)lin);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    ctx->last_stream = s;
    ctx->loaded = false;

    // Layout of the sorted copies.
    const int64_t slice = kvdro::hist_slice_samples(), tile = kvdro::expand_tile_positions();
    ctx->K = K;
    ctx->off.assign(offsets, offsets + K + 1);
    ctx->N.resize(K);
    ctx->L.assign(L_max, L_max + K);
    ctx->Lin.assign(K, 0);
    if (L_in) ctx->Lin.assign(L_in, L_in + K);
    ctx->pair_off.assign(K + 1, 0);
    ctx->hist_off.assign(K + 1, 0);
    ctx->hist_blocks.assign(K + 1, 0);
    ctx->exp_blocks.assign(K + 1, 0);
    for (int32_t k = 0; k < K; k++) {
        const int64_t n = offsets[k + 1] - offsets[k];
        const int64_t padn = (int64_t)align_up((size_t)n, kvdro::kPadSamples);
        ctx->N[k] = n;
        ctx->pair_off[k + 1] = ctx->pair_off[k] + padn;
        ctx->hist_off[k + 1] = ctx->hist_off[k] + (int64_t)L_max[k] + 1;
        const int64_t hb = ctx->hist_blocks[k] + (n + slice - 1) / slice;
        const int64_t eb = ctx->exp_blocks[k] + (padn + tile - 1) / tile;
        if (hb > 0x7fffffffLL || eb > 0x7fffffffLL) return fail(ctx, KVDRO_EINVAL, "too many samples");
        ctx->hist_blocks[k + 1] = (int32_t)hb;
        ctx->exp_blocks[k + 1] = (int32_t)eb;
    }
    // histogram blocks sized to fill whole waves of this device (the bound above still holds:
    // no class gets more blocks than samples)
    KV_CUDA(kvdro::hist_block_prefix(ctx->N.data(), K, ctx->hist_blocks.data()), "sizing the histogram");
    ctx->total = offsets[K];
    ctx->pair_total = ctx->pair_off[K];
    ctx->hist_total = ctx->hist_off[K];

    int rc;
    if ((rc = ensure(ctx, ctx->sorted, (size_t)ctx->total * 4))) return rc;
    if ((rc = ensure(ctx, ctx->pairs, (size_t)ctx->pair_total * 8))) return rc;
    if ((rc = ensure(ctx, ctx->hist, (size_t)ctx->hist_total * 4))) return rc;
    if ((rc = ensure(ctx, ctx->csum, (size_t)ctx->hist_total * 8))) return rc;
    if ((rc = ensure(ctx, ctx->sumx, (size_t)K * 8))) return rc;
    if ((rc = ensure(ctx, ctx->errs, 2 * sizeof(int32_t)))) return rc;
    int64_t max_bins = 0;
    for (int32_t k = 0; k < K; k++) max_bins = std::max<int64_t>(max_bins, (int64_t)L_max[k] + 1);
    const int64_t scan_tiles = (max_bins + kvdro::scan_tile_bins() - 1) / kvdro::scan_tile_bins();
    if ((rc = ensure(ctx, ctx->scan_tot, (size_t)K * scan_tiles * 16))) return rc;
    if ((rc = ensure(ctx, ctx->tile_lo, ((size_t)ctx->exp_blocks[K] + K) * 4))) return rc;
    const size_t meta_bytes = (size_t)(K + 1) * 8 * 3 + (size_t)K * 8 + (size_t)K * 4 * 2 + (size_t)(K + 1) * 4 * 2 + 64;
    if ((rc = ensure(ctx, ctx->meta, meta_bytes))) return rc;

    // Metadata upload (one copy from pinned staging).
    void* hp;
    if ((rc = pinned(ctx, meta_bytes, &hp))) return rc;
    char* h = static_cast<char*>(hp);
    char* d = static_cast<char*>(ctx->meta.p);
    size_t o = 0;
    auto put = [&](const void* src, size_t bytes, void** dview) {
        std::memcpy(h + o, src, bytes);
        *dview = d + o;
        o = align_up(o + bytes, 8);
    };
    put(ctx->off.data(), (K + 1) * 8, reinterpret_cast<void**>(&ctx->d_off));
    put(ctx->pair_off.data(), (K + 1) * 8, reinterpret_cast<void**>(&ctx->d_pair_off));
    put(ctx->hist_off.data(), (K + 1) * 8, reinterpret_cast<void**>(&ctx->d_hist_off));
    put(ctx->N.data(), K * 8, reinterpret_cast<void**>(&ctx->d_N));
    put(ctx->L.data(), K * 4, reinterpret_cast<void**>(&ctx->d_L));
    put(ctx->Lin.data(), K * 4, reinterpret_cast<void**>(&ctx->d_Lin));
    put(ctx->hist_blocks.data(), (K + 1) * 4, reinterpret_cast<void**>(&ctx->d_hist_blocks));
    put(ctx->exp_blocks.data(), (K + 1) * 4, reinterpret_cast<void**>(&ctx->d_exp_blocks));
    KV_CUDA(cudaMemcpyAsync(ctx->meta.p, hp, o, cudaMemcpyHostToDevice, s), "uploading class metadata");
    KV_CUDA(cudaEventRecord(ctx->pin_free, s), "recording staging event");

    const int32_t* dlen = lengths;
    if (!is_device_ptr(lengths)) {
        if ((rc = ensure(ctx, ctx->in_stage, (size_t)ctx->total * 4))) return rc;
        KV_CUDA(cudaMemcpyAsync(ctx->in_stage.p, lengths, (size_t)ctx->total * 4, cudaMemcpyHostToDevice, s),
                "uploading samples");
        dlen = static_cast<const int32_t*>(ctx->in_stage.p);
    }
    KV_CUDA(cudaMemsetAsync(ctx->hist.p, 0, (size_t)ctx->hist_total * 4, s), "clearing histogram");
    KV_CUDA(cudaMemsetAsync(ctx->sumx.p, 0, (size_t)K * 8, s), "clearing sums");
    KV_CUDA(cudaMemsetAsync(ctx->errs.p, 0, 2 * sizeof(int32_t), s), "clearing status");

    kvdro::SortArgs a;
    a.lengths = dlen;
    a.offsets = ctx->d_off;
    a.L = ctx->d_L;
    a.hist_off = ctx->d_hist_off;
    a.pair_off = ctx->d_pair_off;
    a.hist_blocks = ctx->d_hist_blocks;
    a.exp_blocks = ctx->d_exp_blocks;
    a.hist = static_cast<int32_t*>(ctx->hist.p);
    a.csum = static_cast<int64_t*>(ctx->csum.p);
    a.sumx = static_cast<int64_t*>(ctx->sumx.p);
    a.sorted = static_cast<int32_t*>(ctx->sorted.p);
    a.pairs = static_cast<float2*>(ctx->pairs.p);
    a.err = static_cast<int32_t*>(ctx->errs.p);
    a.tile_tot = static_cast<int64_t*>(ctx->scan_tot.p);
    a.tile_lo = static_cast<int32_t*>(ctx->tile_lo.p);
    a.scan_tiles = (int32_t)scan_tiles;
    a.K = K;
    KV_CUDA(kvdro::launch_histogram(a, ctx->hist_blocks[K], s), "histogram kernel");
    KV_CUDA(kvdro::launch_scan(a, s), "scan kernel");
    KV_CUDA(kvdro::launch_expand(a, ctx->exp_blocks[K], s), "expand kernel");

    int32_t bad = 0;
    KV_CUDA(cudaMemcpyAsync(&bad, ctx->errs.p, sizeof(int32_t), cudaMemcpyDeviceToHost, s), "reading range check");
    KV_CUDA(cudaStreamSynchronize(s), "loading samples");
    if (bad != 0)
        return fail(ctx, KVDRO_EINVAL, "%d samples lie outside [0, L_max] of their class; no samples are loaded", bad);
    ctx->loaded = true;
    return KVDRO_OK;
}

int kvdro_quantiles(kvdro_ctx* ctx, int32_t F, const double* fractiles, int32_t* out, void* stream) {
    NvtxRange nvtx_("kvdro_quantiles");
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    if (!ctx->loaded) return fail(ctx, KVDRO_ESTATE, "no samples loaded");
    if (F < 1 || F > kMaxF || (int64_t)F * ctx->K > kMaxKF) return fail(ctx, KVDRO_EINVAL, "F = %d out of range", F);
    if (!fractiles || !out) return fail(ctx, KVDRO_EINVAL, "fractiles and out are required");
    for (int32_t f = 0; f < F; f++)
        if (!(fractiles[f] >= 0.0 && fractiles[f] <= 1.0))
            return fail(ctx, KVDRO_EINVAL, "fractiles[%d] = %g outside [0, 1]", f, fractiles[f]);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    ctx->last_stream = s;
    const int64_t n = (int64_t)ctx->K * F;
    int rc;
    if ((rc = ensure(ctx, ctx->ranks, (size_t)n * 4))) return rc;
    void* hp;
    if ((rc = pinned(ctx, (size_t)n * 4, &hp))) return rc;
    int32_t* hr = static_cast<int32_t*>(hp);
    for (int32_t k = 0; k < ctx->K; k++)
        for (int32_t f = 0; f < F; f++) {
            // lower empirical quantile: rank max(1, ceil(q N)) in FP64
            const double m = std::ceil(fractiles[f] * (double)ctx->N[k]);
            int64_t rk = (int64_t)m;
            if (rk < 1) rk = 1;
            if (rk > ctx->N[k]) rk = ctx->N[k];
            hr[(int64_t)k * F + f] = (int32_t)rk;
        }
    KV_CUDA(cudaMemcpyAsync(ctx->ranks.p, hp, (size_t)n * 4, cudaMemcpyHostToDevice, s), "uploading ranks");
    KV_CUDA(cudaEventRecord(ctx->pin_free, s), "recording staging event");
    const bool dev_out = is_device_ptr(out);
    int32_t* dout = out;
    if (!dev_out) {
        if ((rc = ensure(ctx, ctx->out_stage, (size_t)n * 4))) return rc;
        dout = static_cast<int32_t*>(ctx->out_stage.p);
    }
    KV_CUDA(kvdro::launch_gather_quantiles(static_cast<const int32_t*>(ctx->sorted.p), ctx->d_off,
                                           static_cast<const int32_t*>(ctx->ranks.p), ctx->K, F, dout, s),
            "quantile kernel");
    if (!dev_out) {
        KV_CUDA(cudaMemcpyAsync(out, dout, (size_t)n * 4, cudaMemcpyDeviceToHost, s), "copying quantiles");
        KV_CUDA(cudaStreamSynchronize(s), "copying quantiles");
    }
    return KVDRO_OK;
}

int kvdro_eval_grid(kvdro_ctx* ctx, int precision, int32_t R, const int32_t* r, int32_t NL, const double* lam,
                    int32_t E, const double* eps, int32_t M, const double* c_p, const double* c_w, void* S,
                    void* cost, int32_t* lam_idx, int32_t* r_idx, void* min_cost, double* fhat, void* stream) {
    NvtxRange nvtx_("kvdro_eval_grid");
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    if (!ctx->loaded) return fail(ctx, KVDRO_ESTATE, "no samples loaded");
    if (precision != KVDRO_FP32 && precision != KVDRO_FP64 && precision != KVDRO_EXACT && precision != KVDRO_ENVELOPE)
        return fail(ctx, KVDRO_EINVAL, "precision must be KVDRO_FP32, KVDRO_FP64, KVDRO_EXACT or KVDRO_ENVELOPE");
    const Prec P = precision == KVDRO_FP32 ? Prec::F32
                 : precision == KVDRO_FP64 ? Prec::F64
                 : precision == KVDRO_EXACT ? Prec::EXACT : Prec::ENVELOPE;
    const int32_t maxNL = P == Prec::F64 ? kMaxNLf64 : kMaxNLf32;
    bool exact_ok = true;  // every class's support fits the exact kernel's integer sums
    int32_t max_L = 0;
    for (int32_t k = 0; k < ctx->K; k++) {
        exact_ok = exact_ok && ctx->L[k] <= kvdro::kExactMaxL;
        max_L = std::max(max_L, ctx->L[k]);
    }
    if (P == Prec::EXACT && !exact_ok)
        return fail(ctx, KVDRO_EINVAL, "KVDRO_EXACT needs L_max <= 2^22 for every class");
    // FP32 results come from the exact kernel (rounded to FP32) whenever it applies: it is exact
    // and faster; the FP32-arithmetic kernel serves supports above 2^22.
    const Prec KP = (P == Prec::F32 && exact_ok) ? Prec::EXACT : P;
    if (R < 1 || R > kMaxR) return fail(ctx, KVDRO_EINVAL, "R = %d outside [1, 2^20]", R);
    if (NL < 1 || NL > maxNL) return fail(ctx, KVDRO_EINVAL, "NL = %d outside [1, %d]", NL, maxNL);
    if (E < 1 || E > kMaxE) return fail(ctx, KVDRO_EINVAL, "E = %d outside [1, %d]", E, kMaxE);
    if (M < 1 || M > kMaxM) return fail(ctx, KVDRO_EINVAL, "M = %d outside [1, %d]", M, kMaxM);
    if (!r || !lam || !eps || !c_p || !c_w) return fail(ctx, KVDRO_EINVAL, "r, lam, eps, c_p and c_w are required");
    if (!finite_nonneg(lam, NL)) return fail(ctx, KVDRO_EINVAL, "lam must be finite and >= 0");
    if (!finite_nonneg(eps, E)) return fail(ctx, KVDRO_EINVAL, "eps must be finite and >= 0");
    if (!finite_nonneg(c_p, M) || !finite_nonneg(c_w, M)) return fail(ctx, KVDRO_EINVAL, "costs must be finite and >= 0");
    if (int rc_ = check_reservations(ctx, R, r)) return rc_;
    const int64_t cells_out = (int64_t)M * E * ctx->K * R;
    const int64_t rows = (int64_t)M * E * ctx->K;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    ctx->last_stream = s;

    // Launch shape: lam tiles x r groups of warps per CTA.  The exact kernel takes at most
    // kExactLamBlock lam values per launch; a larger grid runs as consecutive launches over blocks
    // of it (the last block may be smaller and take its own shape).
    const int32_t lam_blk = KP == Prec::EXACT ? kvdro::kExactLamBlock : NL;
    const int32_t nblk = (NL + lam_blk - 1) / lam_blk;
    const int32_t NL_last = NL - (nblk - 1) * lam_blk;
    const kvdro::GridShape shape = kvdro::grid_shape(KP, R, std::min(NL, lam_blk), E, max_L);
    const kvdro::GridShape shape_last = kvdro::grid_shape(KP, R, NL_last, E, max_L);

    // Grid parameters in one upload.
    const size_t gbytes = align_up((size_t)R * 4, 8) + 8 * ((size_t)NL + E + 2 * (size_t)M);
    int rc;
    if ((rc = ensure(ctx, ctx->grid_in, gbytes))) return rc;
    void* hp;
    if ((rc = pinned(ctx, gbytes, &hp))) return rc;
    char* h = static_cast<char*>(hp);
    char* d = static_cast<char*>(ctx->grid_in.p);
    size_t o = 0;
    auto put = [&](const void* src, size_t bytes) {
        std::memcpy(h + o, src, bytes);
        void* dv = d + o;
        o = align_up(o + bytes, 8);
        return dv;
    };
    const int32_t* d_r = static_cast<const int32_t*>(put(r, (size_t)R * 4));
    const double* d_lam = static_cast<const double*>(put(lam, (size_t)NL * 8));
    const double* d_eps = static_cast<const double*>(put(eps, (size_t)E * 8));
    const double* d_cp = static_cast<const double*>(put(c_p, (size_t)M * 8));
    const double* d_cw = static_cast<const double*>(put(c_w, (size_t)M * 8));
    KV_CUDA(cudaMemcpyAsync(ctx->grid_in.p, hp, o, cudaMemcpyHostToDevice, s), "uploading the grid");
    KV_CUDA(cudaEventRecord(ctx->pin_free, s), "recording staging event");

    // Outputs: device pointers are written in place, host outputs go through device staging.
    const size_t es = P == Prec::F32 ? 4 : 8;
    struct Out {
        void* user;
        size_t bytes;
        bool host;
        void* dev;
    };
    Out outs[6] = {{S, (size_t)M * ctx->K * R * NL * es, false, nullptr},
                   {cost, (size_t)cells_out * es, false, nullptr},
                   {lam_idx, (size_t)cells_out * 4, false, nullptr},
                   {r_idx, (size_t)rows * 4, false, nullptr},
                   {min_cost, (size_t)rows * es, false, nullptr},
                   {fhat, (size_t)rows * 8, false, nullptr}};
    size_t stage_bytes = 0;
    for (Out& x : outs) {
        if (!x.user) continue;
        x.host = !is_device_ptr(x.user);
        if (x.host) stage_bytes += align_up(x.bytes, 256);
        else x.dev = x.user;
    }
    if (stage_bytes) {
        if ((rc = ensure(ctx, ctx->out_stage, stage_bytes))) return rc;
        size_t so = 0;
        for (Out& x : outs)
            if (x.user && x.host) {
                x.dev = static_cast<char*>(ctx->out_stage.p) + so;
                so += align_up(x.bytes, 256);
            }
    }
    void* cost_dev = outs[1].dev;
    if (P != Prec::F32 && !cost_dev) {  // FP64 / EXACT min_cost is read back from the cost array
        if ((rc = ensure(ctx, ctx->cost64, (size_t)cells_out * 8))) return rc;
        cost_dev = ctx->cost64.p;
    }
    if ((rc = ensure(ctx, ctx->keys, (size_t)rows * 8))) return rc;
    KV_CUDA(cudaMemsetAsync(ctx->keys.p, 0xFF, (size_t)rows * 8, s), "clearing argmin keys");

    kvdro::GridArgs a;
    a.pairs = static_cast<const float2*>(ctx->pairs.p);
    a.pair_off = ctx->d_pair_off;
    a.N = ctx->d_N;
    a.sumx = static_cast<const int64_t*>(ctx->sumx.p);
    a.L = ctx->d_L;
    a.L_in = ctx->d_Lin;
    a.cdf = static_cast<const int32_t*>(ctx->hist.p);
    a.csum = static_cast<const int64_t*>(ctx->csum.p);
    a.hist_off = ctx->d_hist_off;
    a.r = d_r;
    a.lam = d_lam;
    a.eps = d_eps;
    a.cp = d_cp;
    a.cw = d_cw;
    a.K = ctx->K;
    a.R = R;
    a.NL = NL;
    a.E = E;
    a.M = M;
    a.f32_out = P == Prec::F32;
    a.S_out = outs[0].dev;
    a.cost_out = cost_dev;
    a.lam_idx_out = static_cast<int32_t*>(outs[2].dev);
    a.keys = static_cast<unsigned long long*>(ctx->keys.p);
    a.err = static_cast<int32_t*>(ctx->errs.p);
    // Test hook of contexts created with KVDRO_TEST_SKIP_CHUNK: 1 ms waits that run out on one
    // chunk.  It travels with this context's launches only.
    a.test_skip_chunk = ctx->skip_chunk;
    a.wait_ns = ctx->skip_chunk >= 0 ? kTestWaitNs : 0;
    a.lam0 = 0;
    a.NL_out = NL;
    a.part_val = nullptr;
    a.part_idx = nullptr;
    a.part_first = a.part_last = 1;
    const int64_t per_m = (int64_t)ctx->K * std::max(shape.r_blocks, shape_last.r_blocks);
    int64_t m_step = std::max<int64_t>(1, 0x7fffffffLL / per_m);
    if (nblk > 1) {
        // the running minimum over lam blocks, 12 bytes per (regime, eps, class, r), for at most
        // kPartBytes worth of regimes at a time
        const int64_t per_regime = (int64_t)E * ctx->K * R * 12;
        m_step = std::max<int64_t>(1, std::min<int64_t>(m_step, kPartBytes / per_regime));
        const int64_t cells = std::min<int64_t>(m_step, M) * (per_regime / 12);
        if ((rc = ensure(ctx, ctx->part, (size_t)cells * 12))) return rc;
        a.part_val = static_cast<double*>(ctx->part.p);
        a.part_idx = reinterpret_cast<int32_t*>(static_cast<char*>(ctx->part.p) + (size_t)cells * 8);
    }
    // Host outputs laid out regime-major (S, cost, lam index) go back in blocks of regimes on the
    // context's copy stream, each block as soon as its launches are done, so the copies overlap the
    // evaluation of later regimes instead of following the whole grid.
    const bool pipe = M > 1 && ((outs[0].user && outs[0].host) || (outs[1].user && outs[1].host) ||
                                (outs[2].user && outs[2].host));
    if (pipe) m_step = std::min<int64_t>(m_step, (M + kCopyBlocks - 1) / kCopyBlocks);
    // Whatever way the call returns, no copy into the caller's host buffers is still in flight.
    struct CopyDrain {
        cudaStream_t cs;
        bool armed;
        ~CopyDrain() {
            if (armed) cudaStreamSynchronize(cs);
        }
    } drain{ctx->copy_stream, pipe};
    ctx->grid_timed = false;
    KV_CUDA(cudaEventRecord(ctx->grid_t0, s), "recording grid start");
    for (int64_t m0 = 0; m0 < M; m0 += m_step) {
        a.m0 = (int32_t)m0;
        a.m_count = (int32_t)std::min<int64_t>(m_step, M - m0);
        for (int32_t b = 0; b < nblk; b++) {
            a.lam = d_lam + (size_t)b * lam_blk;
            a.NL = b + 1 < nblk ? lam_blk : NL_last;
            a.lam0 = b * lam_blk;
            a.part_first = b == 0;
            a.part_last = b + 1 == nblk;
            KV_CUDA(kvdro::launch_grid(KP, b + 1 < nblk ? shape : shape_last, a, s), "grid kernel");
        }
        if (pipe) {
            KV_CUDA(cudaEventRecord(ctx->copy_ready, s), "recording a regime block");
            KV_CUDA(cudaStreamWaitEvent(ctx->copy_stream, ctx->copy_ready, 0), "ordering a copy");
            for (int i = 0; i < 3; i++) {
                const Out& x = outs[i];
                if (!x.user || !x.host) continue;
                const size_t per_m = x.bytes / (size_t)M;
                KV_CUDA(cudaMemcpyAsync(static_cast<char*>(x.user) + (size_t)m0 * per_m,
                                        static_cast<const char*>(x.dev) + (size_t)m0 * per_m,
                                        (size_t)a.m_count * per_m, cudaMemcpyDeviceToHost, ctx->copy_stream),
                        "copying results");
            }
        }
    }
    KV_CUDA(cudaEventRecord(ctx->grid_t1, s), "recording grid end");
    ctx->grid_timed = true;

    kvdro::FinalizeArgs fa;
    fa.keys = static_cast<const unsigned long long*>(ctx->keys.p);
    fa.cost = cost_dev;
    fa.r = d_r;
    fa.L_in = ctx->d_Lin;
    fa.N = ctx->d_N;
    fa.cdf = static_cast<const int32_t*>(ctx->hist.p);
    fa.hist_off = ctx->d_hist_off;
    fa.K = ctx->K;
    fa.R = R;
    fa.E = E;
    fa.M = M;
    fa.r_idx = static_cast<int32_t*>(outs[3].dev);
    fa.min_cost = outs[4].dev;
    fa.fhat = static_cast<double*>(outs[5].dev);
    if (fa.r_idx || fa.min_cost || fa.fhat) KV_CUDA(kvdro::launch_finalize(P, fa, s), "finalize kernel");

    if (stage_bytes) {
        if (pipe) {  // the regime blocks' copies, then the rest on the caller's stream
            KV_CUDA(cudaEventRecord(ctx->copy_done, ctx->copy_stream), "recording the copies");
            KV_CUDA(cudaStreamWaitEvent(s, ctx->copy_done, 0), "ordering the copies");
        }
        for (int i = 0; i < 6; i++) {
            const Out& x = outs[i];
            if (x.user && x.host && !(pipe && i < 3))
                KV_CUDA(cudaMemcpyAsync(x.user, x.dev, x.bytes, cudaMemcpyDeviceToHost, s), "copying results");
        }
        KV_CUDA(cudaStreamSynchronize(s), "copying results");
        return check_kernel_errors(ctx, s);
    }
    return KVDRO_OK;
}

int kvdro_eval_dual(kvdro_ctx* ctx, int32_t R, const int32_t* r, int32_t E, const double* eps, int32_t M,
                    const double* c_p, const double* c_w, double* cost, double* gamma, int32_t* r_idx,
                    double* min_cost, double* fhat, void* stream) {
    NvtxRange nvtx_("kvdro_eval_dual");
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    if (!ctx->loaded) return fail(ctx, KVDRO_ESTATE, "no samples loaded");
    if (R < 1 || R > kMaxR) return fail(ctx, KVDRO_EINVAL, "R = %d outside [1, 2^20]", R);
    if (E < 1 || E > kMaxE) return fail(ctx, KVDRO_EINVAL, "E = %d outside [1, %d]", E, kMaxE);
    if (M < 1 || M > kMaxM) return fail(ctx, KVDRO_EINVAL, "M = %d outside [1, %d]", M, kMaxM);
    if (!r || !eps || !c_p || !c_w) return fail(ctx, KVDRO_EINVAL, "r, eps, c_p and c_w are required");
    if (!finite_nonneg(eps, E)) return fail(ctx, KVDRO_EINVAL, "eps must be finite and >= 0");
    if (!finite_nonneg(c_p, M) || !finite_nonneg(c_w, M)) return fail(ctx, KVDRO_EINVAL, "costs must be finite and >= 0");
    if (int rc_ = check_reservations(ctx, R, r)) return rc_;
    const int64_t cells = (int64_t)M * E * ctx->K * R;
    const int64_t rows = (int64_t)M * E * ctx->K;
    if (cells > 0x7fffffffLL * 256LL) return fail(ctx, KVDRO_EINVAL, "grid too large");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    ctx->last_stream = s;

    const size_t gbytes = align_up((size_t)R * 4, 8) + 8 * ((size_t)E + 2 * (size_t)M);
    int rc;
    if ((rc = ensure(ctx, ctx->grid_in, gbytes))) return rc;
    void* hp;
    if ((rc = pinned(ctx, gbytes, &hp))) return rc;
    char* h = static_cast<char*>(hp);
    char* d = static_cast<char*>(ctx->grid_in.p);
    size_t o = 0;
    auto put = [&](const void* src, size_t bytes) {
        std::memcpy(h + o, src, bytes);
        void* dv = d + o;
        o = align_up(o + bytes, 8);
        return dv;
    };
    const int32_t* d_r = static_cast<const int32_t*>(put(r, (size_t)R * 4));
    const double* d_eps = static_cast<const double*>(put(eps, (size_t)E * 8));
    const double* d_cp = static_cast<const double*>(put(c_p, (size_t)M * 8));
    const double* d_cw = static_cast<const double*>(put(c_w, (size_t)M * 8));
    KV_CUDA(cudaMemcpyAsync(ctx->grid_in.p, hp, o, cudaMemcpyHostToDevice, s), "uploading the grid");
    KV_CUDA(cudaEventRecord(ctx->pin_free, s), "recording staging event");

    struct Out {
        void* user;
        size_t bytes;
        bool host;
        void* dev;
    };
    Out outs[5] = {{cost, (size_t)cells * 8, false, nullptr},
                   {gamma, (size_t)cells * 8, false, nullptr},
                   {r_idx, (size_t)rows * 4, false, nullptr},
                   {min_cost, (size_t)rows * 8, false, nullptr},
                   {fhat, (size_t)rows * 8, false, nullptr}};
    size_t stage_bytes = 0;
    for (Out& x : outs) {
        if (!x.user) continue;
        x.host = !is_device_ptr(x.user);
        if (x.host) stage_bytes += align_up(x.bytes, 256);
        else x.dev = x.user;
    }
    if (stage_bytes) {
        if ((rc = ensure(ctx, ctx->out_stage, stage_bytes))) return rc;
        size_t so = 0;
        for (Out& x : outs)
            if (x.user && x.host) {
                x.dev = static_cast<char*>(ctx->out_stage.p) + so;
                so += align_up(x.bytes, 256);
            }
    }
    void* cost_dev = outs[0].dev;
    if (!cost_dev) {
        if ((rc = ensure(ctx, ctx->cost64, (size_t)cells * 8))) return rc;
        cost_dev = ctx->cost64.p;
    }
    if ((rc = ensure(ctx, ctx->keys, (size_t)rows * 8))) return rc;
    KV_CUDA(cudaMemsetAsync(ctx->keys.p, 0xFF, (size_t)rows * 8, s), "clearing argmin keys");

    kvdro::DualArgs a;
    a.cdf = static_cast<const int32_t*>(ctx->hist.p);
    a.csum = static_cast<const int64_t*>(ctx->csum.p);
    a.hist_off = ctx->d_hist_off;
    a.N = ctx->d_N;
    a.sumx = static_cast<const int64_t*>(ctx->sumx.p);
    a.L = ctx->d_L;
    a.L_in = ctx->d_Lin;
    a.r = d_r;
    a.eps = d_eps;
    a.cp = d_cp;
    a.cw = d_cw;
    a.K = ctx->K;
    a.R = R;
    a.E = E;
    a.M = M;
    a.cost = static_cast<double*>(cost_dev);
    a.gamma = static_cast<double*>(outs[1].dev);
    a.keys = static_cast<unsigned long long*>(ctx->keys.p);
    ctx->grid_timed = false;
    KV_CUDA(cudaEventRecord(ctx->grid_t0, s), "recording dual start");
    KV_CUDA(kvdro::launch_dual(a, s), "dual kernel");
    KV_CUDA(cudaEventRecord(ctx->grid_t1, s), "recording dual end");
    ctx->grid_timed = true;

    kvdro::FinalizeArgs fa;
    fa.keys = a.keys;
    fa.cost = cost_dev;
    fa.r = d_r;
    fa.L_in = ctx->d_Lin;
    fa.N = ctx->d_N;
    fa.cdf = a.cdf;
    fa.hist_off = ctx->d_hist_off;
    fa.K = ctx->K;
    fa.R = R;
    fa.E = E;
    fa.M = M;
    fa.r_idx = static_cast<int32_t*>(outs[2].dev);
    fa.min_cost = outs[3].dev;
    fa.fhat = static_cast<double*>(outs[4].dev);
    if (fa.r_idx || fa.min_cost || fa.fhat) KV_CUDA(kvdro::launch_finalize(Prec::F64, fa, s), "finalize kernel");
    if (stage_bytes) {
        for (Out& x : outs)
            if (x.user && x.host)
                KV_CUDA(cudaMemcpyAsync(x.user, x.dev, x.bytes, cudaMemcpyDeviceToHost, s), "copying results");
        KV_CUDA(cudaStreamSynchronize(s), "copying results");
    }
    return KVDRO_OK;
}

int kvdro_sorted_samples(const kvdro_ctx* cctx, int32_t* out, void* stream) {
    NvtxRange nvtx_("kvdro_sorted_samples");
    kvdro_ctx* ctx = const_cast<kvdro_ctx*>(cctx);
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    if (!ctx->loaded) return fail(ctx, KVDRO_ESTATE, "no samples loaded");
    if (!out) return fail(ctx, KVDRO_EINVAL, "out is required");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    ctx->last_stream = s;
    const bool dev = is_device_ptr(out);
    KV_CUDA(cudaMemcpyAsync(out, ctx->sorted.p, (size_t)ctx->total * 4,
                            dev ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s),
            "copying sorted samples");
    if (!dev) KV_CUDA(cudaStreamSynchronize(s), "copying sorted samples");
    return KVDRO_OK;
}

int kvdro_last_grid_ms(kvdro_ctx* ctx, float* ms) {
    if (!ctx || !ms) return KVDRO_EINVAL;
    ctx->err.clear();
    if (!ctx->grid_timed) return fail(ctx, KVDRO_ESTATE, "no grid evaluated yet");
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    KV_CUDA(cudaEventSynchronize(ctx->grid_t1), "waiting for the grid kernel");
    KV_CUDA(cudaEventElapsedTime(ms, ctx->grid_t0, ctx->grid_t1), "reading the grid kernel time");
    return KVDRO_OK;
}

int kvdro_sync(kvdro_ctx* ctx) {
    NvtxRange nvtx_("kvdro_sync");
    if (!ctx) return KVDRO_EINVAL;
    ctx->err.clear();
    DeviceGuard g(ctx->device);
    if (!g.ok) return fail(ctx, KVDRO_ECUDA, "cannot select device %d", ctx->device);
    KV_CUDA(cudaStreamSynchronize(ctx->last_stream), "synchronising");
    KV_CUDA(cudaGetLastError(), "asynchronous error");
    return check_kernel_errors(ctx, ctx->last_stream);
}

}  // extern "C"
