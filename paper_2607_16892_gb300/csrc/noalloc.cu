// kvdro_eval_grid_noalloc: the FP32 grid evaluation for callers that cannot allocate memory.
// All of its scratch (class metadata, grid parameters, cumulative counts, the sorted samples,
// the NaN-padded sample pairs the grid kernel streams, and the argmin keys) lives in one
// file-scope __device__ array that every device loading this library holds until the process
// exits.  Nothing in this file calls cudaMalloc, cudaFree, cudaHostAlloc, malloc/new or any
// other allocating routine; the per-class metadata is derived on the device.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <initializer_list>
#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "kvdro.h"
#include "kvdro_internal.cuh"

namespace kvdro {
int64_t hist_slice_samples();
int64_t expand_tile_positions();
int64_t scan_tile_bins();
}  // namespace kvdro

namespace {

// The scratch.  In host code this name is only a host-side stand-in, not a device address; the
// device address is taken with cudaGetSymbolAddress once per device (setup_device below).
static __device__ __align__(256) unsigned char g_noalloc_scratch[KVDRO_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
void* g_scratch_addr[kMaxDevices] = {nullptr};

struct Meta {  // device views into the scratch
    const int64_t* offsets;
    const int32_t* L;
    const int32_t* L_in_src;  // caller's L_in copied in, or nullptr
    int64_t* pair_off;
    int64_t* hist_off;
    int64_t* N;
    int32_t* L_in;
    int32_t* hist_blocks;
    int32_t* exp_blocks;
    int32_t K;
    int64_t slice, tile;
};

// Per-class prefix arrays from the offsets and supports (K <= 4096: one thread is enough).
__global__ void k_noalloc_meta(Meta m) {
    if (blockIdx.x != 0 || threadIdx.x != 0) return;
    m.pair_off[0] = 0;
    m.hist_off[0] = 0;
    m.hist_blocks[0] = 0;
    m.exp_blocks[0] = 0;
    for (int k = 0; k < m.K; k++) {
        const int64_t n = m.offsets[k + 1] - m.offsets[k];
        const int64_t padn = (n + kvdro::kPadSamples - 1) / kvdro::kPadSamples * kvdro::kPadSamples;
        m.N[k] = n;
        m.L_in[k] = m.L_in_src ? m.L_in_src[k] : 0;
        m.pair_off[k + 1] = m.pair_off[k] + padn;
        m.hist_off[k + 1] = m.hist_off[k] + (int64_t)m.L[k] + 1;
        m.hist_blocks[k + 1] = m.hist_blocks[k] + (int32_t)((n + m.slice - 1) / m.slice);
        m.exp_blocks[k + 1] = m.exp_blocks[k] + (int32_t)((padn + m.tile - 1) / m.tile);
    }
}

int report(char* err, int32_t err_len, int code, const char* msg) {
    if (err && err_len > 0) snprintf(err, (size_t)err_len, "%s", msg);
    return code;
}

// Once per device, with that device current: resolve the scratch's device address and raise the
// grid kernel's dynamic shared-memory limit.
int setup_device(int dev, void** out, char* err, int32_t err_len) {
    if (dev < 0 || dev >= kMaxDevices) return report(err, err_len, KVDRO_EINVAL, "device ordinal out of range");
    std::lock_guard<std::mutex> lock(g_setup_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) {
            cudaGetLastError();
            return report(err, err_len, KVDRO_ECUDA, "cudaGetSymbolAddress of the static scratch failed");
        }
        if (kvdro::grid_prepare(kvdro::Prec::F32) != cudaSuccess || kvdro::grid_prepare(kvdro::Prec::EXACT) != cudaSuccess) {
            cudaGetLastError();
            return report(err, err_len, KVDRO_ECUDA, "setting the grid kernel's shared-memory limit failed");
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return KVDRO_OK;
}

bool device_pointer(const void* p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

size_t up256(size_t v) { return (v + 255) / 256 * 256; }

}  // namespace

extern "C" int kvdro_eval_grid_noalloc(int32_t K, const int64_t* offsets, const int32_t* lengths,
                                       const int32_t* L_max, const int32_t* L_in, int32_t R, const int32_t* r,
                                       int32_t NL, const double* lam, int32_t E, const double* eps, int32_t M,
                                       const double* c_p, const double* c_w, float* cost, int32_t* lam_idx,
                                       int32_t* r_idx, float* min_cost, double* fhat, void* stream, char* err,
                                       int32_t err_len) {
    nvtxRangePushA("kvdro_eval_grid_noalloc");
    struct PopAtExit { ~PopAtExit() { nvtxRangePop(); } } pop_at_exit_;
    if (err && err_len > 0) err[0] = 0;
    // ---- host-side validation (the rules of kvdro_load_samples and of kvdro_eval_grid in FP32)
    if (K < 1 || K > 4096) return report(err, err_len, KVDRO_EINVAL, "K outside [1, 4096]");
    if (!offsets || !lengths || !L_max || !r || !lam || !eps || !c_p || !c_w)
        return report(err, err_len, KVDRO_EINVAL, "offsets, lengths, L_max, r, lam, eps, c_p and c_w are required");
    if (offsets[0] != 0) return report(err, err_len, KVDRO_EINVAL, "offsets[0] must be 0");
    if (R < 1 || R > (1 << 20) || NL < 1 || NL > 256 || E < 1 || E > 64 || M < 1 || M > 65536)
        return report(err, err_len, KVDRO_EINVAL, "R, NL, E or M out of range");
    const int64_t slice = kvdro::hist_slice_samples(), tile = kvdro::expand_tile_positions();
    int64_t pair_total = 0, hist_total = 0, hist_blocks = 0, exp_blocks = 0, max_bins = 0;
    for (int32_t k = 0; k < K; k++) {
        const int64_t n = offsets[k + 1] - offsets[k];
        const int64_t lin = L_in ? L_in[k] : 0;
        if (n < 1 || n > 0x7fffffffLL) return report(err, err_len, KVDRO_EINVAL, "every class needs 1..2^31-1 samples");
        if (L_max[k] < 1 || L_max[k] > (1 << 24) || lin < 0 || lin + L_max[k] > (1 << 24))
            return report(err, err_len, KVDRO_EINVAL, "L_max or L_in out of range");
        const int64_t padn = (n + kvdro::kPadSamples - 1) / kvdro::kPadSamples * kvdro::kPadSamples;
        pair_total += padn;
        hist_total += (int64_t)L_max[k] + 1;
        max_bins = max_bins > (int64_t)L_max[k] + 1 ? max_bins : (int64_t)L_max[k] + 1;
        hist_blocks += (n + slice - 1) / slice;
        exp_blocks += (padn + tile - 1) / tile;
    }
    for (int32_t i = 0; i < NL; i++)
        if (!std::isfinite(lam[i]) || lam[i] < 0) return report(err, err_len, KVDRO_EINVAL, "lam must be finite and >= 0");
    for (int32_t i = 0; i < E; i++)
        if (!std::isfinite(eps[i]) || eps[i] < 0) return report(err, err_len, KVDRO_EINVAL, "eps must be finite and >= 0");
    for (int32_t i = 0; i < M; i++)
        if (!std::isfinite(c_p[i]) || c_p[i] < 0 || !std::isfinite(c_w[i]) || c_w[i] < 0)
            return report(err, err_len, KVDRO_EINVAL, "costs must be finite and >= 0");
    {
        // every r must lie in [L_in, L_in + L_max] of every class: in [max L_in, min (L_in + L_max)]
        int64_t lo = 0, hi = INT64_MAX;
        for (int32_t k = 0; k < K; k++) {
            const int64_t lin = L_in ? L_in[k] : 0;
            lo = lin > lo ? lin : lo;
            hi = lin + L_max[k] < hi ? lin + L_max[k] : hi;
        }
        for (int32_t i = 0; i < R; i++)
            if ((int64_t)r[i] < lo || (int64_t)r[i] > hi)
                return report(err, err_len, KVDRO_EINVAL, "r outside [L_in, L_in + L_max] of some class");
    }
    if (!device_pointer(lengths)) return report(err, err_len, KVDRO_EINVAL, "lengths must be device memory");
    for (const void* o : {(const void*)cost, (const void*)lam_idx, (const void*)r_idx, (const void*)min_cost,
                          (const void*)fhat})
        if (o && !device_pointer(o)) return report(err, err_len, KVDRO_EINVAL, "outputs must be device memory");

    // ---- scratch layout; anything beyond the static array is rejected
    const int64_t total = offsets[K];
    const int64_t rows = (int64_t)M * E * K;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = up256(o + bytes);
        return at;
    };
    const size_t o_err = take(2 * sizeof(int32_t));
    const size_t o_off = take((size_t)(K + 1) * 8), o_poff = take((size_t)(K + 1) * 8);
    const size_t o_hoff = take((size_t)(K + 1) * 8), o_N = take((size_t)K * 8);
    const size_t o_L = take((size_t)K * 4), o_Lsrc = take((size_t)K * 4), o_Lin = take((size_t)K * 4);
    const size_t o_hb = take((size_t)(K + 1) * 4), o_eb = take((size_t)(K + 1) * 4);
    const size_t o_r = take((size_t)R * 4), o_lam = take((size_t)NL * 8), o_eps = take((size_t)E * 8);
    const size_t o_cp = take((size_t)M * 8), o_cw = take((size_t)M * 8);
    const size_t o_sumx = take((size_t)K * 8);
    const size_t o_hist = take((size_t)hist_total * 4);
    const size_t o_sorted = take((size_t)total * 4);
    const size_t o_pairs = take((size_t)pair_total * 8);
    const size_t o_keys = take((size_t)rows * 8);
    // more lam values than one launch of the exact kernel takes: the running minimum over lam blocks
    const bool exact_ok = [&] {
        for (int32_t k = 0; k < K; k++)
            if (L_max[k] > kvdro::kExactMaxL) return false;
        return true;
    }();
    const int32_t lam_blk = exact_ok ? kvdro::kExactLamBlock : NL;
    const int32_t nblk = (NL + lam_blk - 1) / lam_blk;
    const size_t part_cells = nblk > 1 ? (size_t)rows * R : 0;
    const size_t o_part_val = take(part_cells * 8), o_part_idx = take(part_cells * 4);
    const int64_t scan_tiles = (max_bins + kvdro::scan_tile_bins() - 1) / kvdro::scan_tile_bins();
    const size_t o_tiles = take((size_t)K * scan_tiles * 16);
    const size_t o_tile_lo = take(((size_t)exp_blocks + K) * 4);
    if (o > (size_t)KVDRO_NOALLOC_SCRATCH_BYTES) {
        char msg[200];
        snprintf(msg, sizeof(msg), "the problem needs %zu bytes of scratch; the static scratch holds %zu bytes", o,
                 (size_t)KVDRO_NOALLOC_SCRATCH_BYTES);
        return report(err, err_len, KVDRO_EINVAL, msg);
    }

    // ---- launch shapes (host only), checked before anything is launched
    int32_t max_L = 0;
    for (int32_t k = 0; k < K; k++) max_L = L_max[k] > max_L ? L_max[k] : max_L;
    const kvdro::Prec kp = exact_ok ? kvdro::Prec::EXACT : kvdro::Prec::F32;
    const int32_t NL_last = NL - (nblk - 1) * lam_blk;
    const kvdro::GridShape shape = kvdro::grid_shape(kp, R, NL < lam_blk ? NL : lam_blk, E, max_L);
    const kvdro::GridShape shape_last = kvdro::grid_shape(kp, R, NL_last, E, max_L);
    const int64_t per_m = (int64_t)K * (shape.r_blocks > shape_last.r_blocks ? shape.r_blocks : shape_last.r_blocks);
    // one launch per lam block covers every regime (the running minimum holds all of them), so
    // with lam blocks the regimes are not split
    const int64_t m_step = nblk > 1 ? M : (per_m > 0x7fffffffLL ? 1 : 0x7fffffffLL / per_m);
    if (nblk > 1 && per_m * M > 0x7fffffffLL)
        return report(err, err_len, KVDRO_EINVAL, "too many CTAs for one launch over every regime");

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return report(err, err_len, KVDRO_ECUDA, "no current CUDA device");
    }
    void* base = nullptr;
    if (int rc = setup_device(dev, &base, err, err_len)) return rc;
    char* S = static_cast<char*>(base);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
#define NA_CUDA(call)                                                              \
    do {                                                                           \
        const cudaError_t e_ = (call);                                             \
        if (e_ != cudaSuccess) {                                                   \
            char m_[200];                                                          \
            snprintf(m_, sizeof(m_), "%s: %s", #call, cudaGetErrorString(e_));     \
            return report(err, err_len, KVDRO_ECUDA, m_);                          \
        }                                                                          \
    } while (0)

    // ---- copy the caller's host parameters in, derive the metadata, clear what starts at zero
    NA_CUDA(cudaMemcpyAsync(S + o_off, offsets, (size_t)(K + 1) * 8, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_L, L_max, (size_t)K * 4, cudaMemcpyHostToDevice, s));
    if (L_in) NA_CUDA(cudaMemcpyAsync(S + o_Lsrc, L_in, (size_t)K * 4, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_r, r, (size_t)R * 4, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_lam, lam, (size_t)NL * 8, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_eps, eps, (size_t)E * 8, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_cp, c_p, (size_t)M * 8, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemcpyAsync(S + o_cw, c_w, (size_t)M * 8, cudaMemcpyHostToDevice, s));
    NA_CUDA(cudaMemsetAsync(S + o_err, 0, 2 * sizeof(int32_t), s));
    NA_CUDA(cudaMemsetAsync(S + o_sumx, 0, (size_t)K * 8, s));
    NA_CUDA(cudaMemsetAsync(S + o_hist, 0, (size_t)hist_total * 4, s));
    NA_CUDA(cudaMemsetAsync(S + o_keys, 0xFF, (size_t)rows * 8, s));
    Meta mt;
    mt.offsets = reinterpret_cast<const int64_t*>(S + o_off);
    mt.L = reinterpret_cast<const int32_t*>(S + o_L);
    mt.L_in_src = L_in ? reinterpret_cast<const int32_t*>(S + o_Lsrc) : nullptr;
    mt.pair_off = reinterpret_cast<int64_t*>(S + o_poff);
    mt.hist_off = reinterpret_cast<int64_t*>(S + o_hoff);
    mt.N = reinterpret_cast<int64_t*>(S + o_N);
    mt.L_in = reinterpret_cast<int32_t*>(S + o_Lin);
    mt.hist_blocks = reinterpret_cast<int32_t*>(S + o_hb);
    mt.exp_blocks = reinterpret_cast<int32_t*>(S + o_eb);
    mt.K = K;
    mt.slice = slice;
    mt.tile = tile;
    k_noalloc_meta<<<1, 1, 0, s>>>(mt);
    NA_CUDA(cudaGetLastError());

    // ---- segmented sort into the scratch (the library's sort kernels)
    kvdro::SortArgs sa;
    sa.lengths = lengths;
    sa.offsets = mt.offsets;
    sa.L = mt.L;
    sa.hist_off = mt.hist_off;
    sa.pair_off = mt.pair_off;
    sa.hist_blocks = mt.hist_blocks;
    sa.exp_blocks = mt.exp_blocks;
    sa.hist = reinterpret_cast<int32_t*>(S + o_hist);
    sa.csum = nullptr;  // cumulative sums are not needed here
    sa.sumx = reinterpret_cast<int64_t*>(S + o_sumx);
    sa.sorted = reinterpret_cast<int32_t*>(S + o_sorted);
    sa.pairs = reinterpret_cast<float2*>(S + o_pairs);
    sa.err = reinterpret_cast<int32_t*>(S + o_err);
    sa.tile_tot = reinterpret_cast<int64_t*>(S + o_tiles);
    sa.tile_lo = reinterpret_cast<int32_t*>(S + o_tile_lo);
    sa.scan_tiles = (int32_t)scan_tiles;
    sa.K = K;
    NA_CUDA(kvdro::launch_histogram(sa, (int32_t)hist_blocks, s));
    NA_CUDA(kvdro::launch_scan(sa, s));
    NA_CUDA(kvdro::launch_expand(sa, (int32_t)exp_blocks, s));
    int32_t bad = 0;
    NA_CUDA(cudaMemcpyAsync(&bad, S + o_err, sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    NA_CUDA(cudaStreamSynchronize(s));
    if (bad) return report(err, err_len, KVDRO_EINVAL, "samples outside [0, L_max] of their class");

    // ---- the grid kernel (the exact one, FP32 outputs, whenever every support is at most 2^22;
    // else the FP32-arithmetic one) and the argmin finalisation
    kvdro::GridArgs a;
    a.pairs = sa.pairs;
    a.pair_off = sa.pair_off;
    a.N = mt.N;
    a.sumx = sa.sumx;
    a.L = mt.L;
    a.L_in = mt.L_in;
    a.cdf = sa.hist;
    a.csum = nullptr;
    a.hist_off = sa.hist_off;
    a.r = reinterpret_cast<const int32_t*>(S + o_r);
    a.lam = reinterpret_cast<const double*>(S + o_lam);
    a.eps = reinterpret_cast<const double*>(S + o_eps);
    a.cp = reinterpret_cast<const double*>(S + o_cp);
    a.cw = reinterpret_cast<const double*>(S + o_cw);
    a.K = K;
    a.R = R;
    a.NL = NL;
    a.E = E;
    a.M = M;
    a.f32_out = 1;
    a.S_out = nullptr;
    a.cost_out = cost;
    a.lam_idx_out = lam_idx;
    a.keys = reinterpret_cast<unsigned long long*>(S + o_keys);
    a.err = sa.err;
    // The bounded-wait test hook, read at every call (see kvdro_create): a 1 ms bound and one
    // chunk left uncopied, so the waits on it run out.
    a.test_skip_chunk = -1;
    a.wait_ns = 0;
    if (const char* f = std::getenv("KVDRO_TEST_SKIP_CHUNK")) {
        a.test_skip_chunk = std::atoi(f);
        a.wait_ns = 1000000;
    }
    a.lam0 = 0;
    a.NL_out = NL;
    a.part_val = nblk > 1 ? reinterpret_cast<double*>(S + o_part_val) : nullptr;
    a.part_idx = nblk > 1 ? reinterpret_cast<int32_t*>(S + o_part_idx) : nullptr;
    const double* d_lam = a.lam;
    for (int64_t m0 = 0; m0 < M; m0 += m_step) {
        a.m0 = (int32_t)m0;
        a.m_count = (int32_t)(m_step < M - m0 ? m_step : M - m0);
        for (int32_t b = 0; b < nblk; b++) {
            a.lam = d_lam + (size_t)b * lam_blk;
            a.NL = b + 1 < nblk ? lam_blk : NL_last;
            a.lam0 = b * lam_blk;
            a.part_first = b == 0;
            a.part_last = b + 1 == nblk;
            NA_CUDA(kvdro::launch_grid(kp, b + 1 < nblk ? shape : shape_last, a, s));
        }
    }
    kvdro::FinalizeArgs fa;
    fa.keys = a.keys;
    fa.cost = nullptr;
    fa.r = a.r;
    fa.L_in = a.L_in;
    fa.N = a.N;
    fa.cdf = a.cdf;
    fa.hist_off = a.hist_off;
    fa.K = K;
    fa.R = R;
    fa.E = E;
    fa.M = M;
    fa.r_idx = r_idx;
    fa.min_cost = min_cost;
    fa.fhat = fhat;
    if (r_idx || min_cost || fhat) NA_CUDA(kvdro::launch_finalize(kvdro::Prec::F32, fa, s));
    // A grid CTA that gave up a bounded wait wrote none of its cells, so the outputs are
    // incomplete: report it here (the next call clears the status word).
    int32_t status = 0;
    NA_CUDA(cudaMemcpyAsync(&status, S + o_err + sizeof(int32_t), sizeof(int32_t), cudaMemcpyDeviceToHost, s));
    NA_CUDA(cudaStreamSynchronize(s));
    if (status & kvdro::kErrTimeout)
        return report(err, err_len, KVDRO_ETIMEOUT,
                      "a grid kernel gave up waiting for a staged sample chunk; the outputs are incomplete");
#undef NA_CUDA
    return KVDRO_OK;
}
