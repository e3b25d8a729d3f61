// The exact dual value of App. A (eq. app_kantorovich, gamma >= 0 not restricted to a grid):
//   cost(eta, eps) = min_{gamma >= 0} g(gamma),  g(gamma) = gamma eps + S(eta, gamma).
// g is convex and piecewise linear in gamma (each sample's supremum is a maximum of lines in
// gamma).  For gamma >= max(c_p, c_w) moving mass never pays and S is the empirical cost, so g
// rises with slope eps and the minimiser lies in [0, max(c_p, c_w)].  One thread per
// (regime, radius, class, reservation) bisects on the sign of the right derivative over the
// bit patterns of the nonnegative doubles (ordered as their values), so the bracket closes to
// two adjacent doubles in at most 63 steps at any scale: a kink at c_w = 1e-250 under c_p = 2
// is found as surely as one near c_p.  Every evaluation of S and of its derivative is O(1) from
// the class's cumulative counts and sums: with mu = min(gamma, c_p), nu = min(gamma, c_w),
// kappa = mu + nu and d = (c_p - mu) L - (c_p + c_w) eta, the samples with a positive excess
// kappa x + d (where U beats V) are x >= t for an integer threshold t, and
//   N S = c_w eta #{x < t} - nu sum_{x < t} x + c_p (L - eta) #{x >= t} - mu sum_{x >= t} (L - x).
#include <float.h>
#include <math.h>

#include "kvdro_internal.cuh"

namespace kvdro {
namespace {

constexpr int kDualThreads = 256;
constexpr int kBisections = 64;  // > 63: enough to close any bracket [0, hi] to adjacent doubles

struct ClassView {
    const int32_t* C;   // cumulative counts, L + 1 entries
    const int64_t* CS;  // cumulative sums
    int64_t N;
    int64_t sumx;
    int32_t L;
};

// count and sum of the samples with x >= t (t clamped to [0, L + 1])
__device__ __forceinline__ void tail(const ClassView& c, int64_t t, int64_t& cnt, int64_t& sum) {
    const int64_t below_n = t >= 1 ? (int64_t)c.C[t - 1] : 0;
    const int64_t below_s = t >= 1 ? c.CS[t - 1] : 0;
    cnt = c.N - below_n;
    sum = c.sumx - below_s;
}

// g(gamma) and its right derivative.
// The samples from the first active point t on, where U beats V: their count and sum.
__device__ __forceinline__ void split_at(const ClassView& c, double eta, double cp, double cw, double gam, double& mu,
                                         double& nu, int64_t& cnt, int64_t& sum) {
    mu = fmin(gam, cp);
    nu = fmin(gam, cw);
    tail(c, first_active(mu + nu, excess_offset(cp, cw, mu, (double)c.L, eta), c.L), cnt, sum);
}

// Sign of the right derivative of g at gamma, eps - (nu' sum_{x < t} x + mu' sum_{x >= t} (L - x)) / N
// with nu' = [gamma < c_w], mu' = [gamma < c_p]: the active set just above gamma is the one at
// gamma up to samples whose excess is exactly zero, which change the value by nothing and the
// slope only at a kink.  Tested as eps N >= the integer sum (eps_n = eps N rounded once), the
// sign is all the bisection needs.
__device__ __forceinline__ bool slope_nonneg(const ClassView& c, double eta, double cp, double cw, double eps_n,
                                             double gam) {
    double mu, nu;
    int64_t cnt, sum;
    split_at(c, eta, cp, cw, gam, mu, nu, cnt, sum);
    const int64_t drop = (gam < cw ? c.sumx - sum : 0) + (gam < cp ? (int64_t)c.L * cnt - sum : 0);
    return eps_n >= (double)drop;
}

// g(gamma) = gamma eps + S(eta, gamma), every sample on its own branch of phi.
__device__ __forceinline__ double value_at(const ClassView& c, double eta, double cp, double cw, double eps,
                                           double gam, double inv_n) {
    double mu, nu;
    int64_t cnt, sum;
    split_at(c, eta, cp, cw, gam, mu, nu, cnt, sum);
    const int64_t below = c.sumx - sum, dist = (int64_t)c.L * cnt - sum;
    return gam * eps + branch_sum(cp, cw, mu, nu, (double)c.L, eta, (double)c.N, cnt, below, dist) * inv_n;
}

__global__ void __launch_bounds__(kDualThreads) k_dual(const DualArgs a) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t total = (int64_t)a.M * a.E * a.K * a.R;
    if (i >= total) return;
    int64_t t = i;
    const int ri = (int)(t % a.R);
    t /= a.R;
    const int k = (int)(t % a.K);
    t /= a.K;
    const int e = (int)(t % a.E);
    const int m = (int)(t / a.E);
    ClassView c;
    c.C = a.cdf + a.hist_off[k];
    c.CS = a.csum + a.hist_off[k];
    c.N = a.N[k];
    c.sumx = a.sumx[k];
    c.L = a.L[k];
    const double cp = a.cp[m], cw = a.cw[m], eps = a.eps[e];
    const double eta = (double)a.r[ri] - (double)a.L_in[k];
    const double inv_n = 1.0 / (double)c.N;
    const double eps_n = eps * (double)c.N;
    double lo = 0.0, hi = fmax(cp, cw);
    double best_g, best_gam;
    if (!slope_nonneg(c, eta, cp, cw, eps_n, lo) && hi > 0.0) {
        long long lb = __double_as_longlong(lo), hb = __double_as_longlong(hi);  // 0 <= lb < hb < 2^63
        for (int it = 0; it < kBisections && hb - lb > 1; it++) {
            const long long mb = lb + (hb - lb) / 2;
            const double mid = __longlong_as_double(mb);
            if (slope_nonneg(c, eta, cp, cw, eps_n, mid)) { hb = mb; hi = mid; }
            else { lb = mb; lo = mid; }
        }
        // g is linear between kinks: the better end of the final bracket is the minimum
        const double g_lo = value_at(c, eta, cp, cw, eps, lo, inv_n), g_hi = value_at(c, eta, cp, cw, eps, hi, inv_n);
        if (g_hi < g_lo) { best_g = g_hi; best_gam = hi; }
        else { best_g = g_lo; best_gam = lo; }
    } else {
        best_g = value_at(c, eta, cp, cw, eps, lo, inv_n);  // g rises from gamma = 0
        best_gam = lo;
    }
    // Every g is at least the empirical cost (1/N) sum Q(eta, x_n): the empirical distribution
    // lies in the ball, and phi >= Q(eta, x) at every gamma.  That bound is exact from integer
    // sums, whereas g near a kink sums branches many orders above it when c_p or c_w is extreme;
    // at eps = 0 it is the value itself.
    {
        const int64_t e_i = (int64_t)a.r[ri] - a.L_in[k];  // eta, in [0, L] on the reservation domain
        int64_t n_up, s_up;
        tail(c, e_i + 1, n_up, s_up);  // the samples above eta
        const double emp = (cw * (double)(e_i * (c.N - n_up) - (c.sumx - s_up)) + cp * (double)(s_up - e_i * n_up)) * inv_n;
        if (best_g < emp) best_g = emp;
    }
    const size_t row = ((size_t)m * a.E + e) * a.K + k;
    if (a.cost) a.cost[row * a.R + ri] = best_g;
    if (a.gamma) a.gamma[row * a.R + ri] = best_gam;
    const unsigned long long key =
        ((unsigned long long)__double_as_longlong(best_g > 0.0 ? best_g : 0.0) & ~0xFFFFFull) | (unsigned long long)ri;
    atomicMin(a.keys + row, key);
}

}  // namespace

cudaError_t launch_dual(const DualArgs& a, cudaStream_t s) {
    const int64_t total = (int64_t)a.M * a.E * a.K * a.R;
    const int64_t blocks = (total + kDualThreads - 1) / kDualThreads;
    if (blocks <= 0 || blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    k_dual<<<(unsigned)blocks, kDualThreads, 0, s>>>(a);
    return cudaGetLastError();
}

}  // namespace kvdro
