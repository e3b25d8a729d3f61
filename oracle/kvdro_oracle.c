/*
 * kvdro_oracle.c -- plain CPU oracle for the Wasserstein-DRO reservation cost.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * reference that the CUDA path is checked against.  Only the tests, the smoke
 * check and the benchmark's CPU-baseline leg may load it.  It shares no code,
 * header, table or helper with the CUDA library, and the library never calls it.
 *
 * What it computes (paper: "Robust KV Cache Management for LLM Serving under
 * Output Token Length Uncertainty", Appendix A, Prop. "Worst-Case Expectation
 * Reformulation"):
 *
 *   eta            = r - L_in                                   (Prop. 2 proof)
 *   Q(eta, xi)     = c_p (xi - eta)^+ + c_w (eta - xi)^+        (Sec. 2.3; App. A Step 1)
 *   phi(x)         = max{ Q(eta,0) - lam x, Q(eta,x), Q(eta,L) - lam (L - x) }
 *                                                               (App. A Step 4, candidates 0, x, L)
 *   S(eta, lam)    = (1/N) sum_n phi(x_n)                       (App. A Step 3, inner mean)
 *
 * The endpoint candidates use the full Q (both (.)^+ terms) at xi = 0 and
 * xi = L.  Inside the paper's domain r in [L_in, L_in + L] (Sec. 2.2) this is
 * the paper's phi^(0) and phi^(L); outside it, it is still the exact supremum.
 * Arithmetic is IEEE double throughout; sums run sequentially in n.  Build
 * with -ffp-contract=off so results are identical on every host.
 *
 * A second evaluator (kvo_envelope_*) regroups the same finite sum by the
 * pieces of the upper envelope of the four affine functions of x that make up
 * phi, using exact integer cumulative counts and sums of the samples.  It is
 * the same quantity, reached with O(1) roundings per cell; the tests pin it
 * against brute force and against the direct sum.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* Q(eta, xi): preemption cost on the shortfall plus memory cost on the excess
 * (Sec. 2.3 "Preemption Cost", "Waste Cost"; App. A Step 1, Q^stoch). */
double kvo_Q(double eta, double xi, double cp, double cw) {
    double over = xi - eta;   /* tokens generated beyond the reservation */
    double under = eta - xi;  /* reserved tokens left unused */
    return cp * (over > 0.0 ? over : 0.0) + cw * (under > 0.0 ? under : 0.0);
}

/* phi: the pointwise supremum over xi in [0, L] of Q(eta, xi) - lam |xi - x|,
 * evaluated at the three candidates the paper lists (App. A Step 4). */
double kvo_phi(double x, double eta, double lam, double cp, double cw, double L) {
    double phi0 = kvo_Q(eta, 0.0, cp, cw) - lam * x;        /* move the sample to xi = 0 */
    double phix = kvo_Q(eta, x, cp, cw);                    /* leave it at xi = x */
    double phiL = kvo_Q(eta, L, cp, cw) - lam * (L - x);    /* move it to xi = L */
    double m = phi0 > phix ? phi0 : phix;
    return m > phiL ? m : phiL;
}

/* S: the empirical mean of phi over one class's samples (App. A Step 3). */
double kvo_mean_sup(const int32_t* x, int64_t n, double eta, double lam, double cp, double cw, double L) {
    double s = 0.0;
    for (int64_t i = 0; i < n; i++) s += kvo_phi((double)x[i], eta, lam, cp, cw, L);
    return s / (double)n;
}

/* ---- direct evaluation of a list of cells, threaded over cells ---------------------------- */

typedef struct {
    const int32_t* samples;
    const int64_t* offsets;
    const int32_t* L;
    const int32_t* L_in;
    const int32_t* r;
    const double* lam;
    const double* cp;
    const double* cw;
    const int32_t* cell_m;
    const int32_t* cell_k;
    const int32_t* cell_r;
    const int32_t* cell_l;
    double* out;
    int64_t begin, end;
} cells_job;

static void* cells_worker(void* arg) {
    cells_job* j = (cells_job*)arg;
    for (int64_t c = j->begin; c < j->end; c++) {
        int m = j->cell_m[c], k = j->cell_k[c];
        const int32_t* x = j->samples + j->offsets[k];
        int64_t n = j->offsets[k + 1] - j->offsets[k];
        double eta = (double)j->r[j->cell_r[c]] - (double)j->L_in[k];
        j->out[c] = kvo_mean_sup(x, n, eta, j->lam[j->cell_l[c]], j->cp[m], j->cw[m], (double)j->L[k]);
    }
    return NULL;
}

static int run_jobs(cells_job* proto, int64_t ncells, int nthreads, void* (*fn)(void*)) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 1024) nthreads = 1024;
    if ((int64_t)nthreads > ncells) nthreads = ncells > 0 ? (int)ncells : 1;
    cells_job* jobs = (cells_job*)malloc(sizeof(cells_job) * (size_t)nthreads);
    pthread_t* th = (pthread_t*)malloc(sizeof(pthread_t) * (size_t)nthreads);
    if (!jobs || !th) { free(jobs); free(th); return -2; }
    int started = 0, rc = 0;
    for (int t = 0; t < nthreads; t++) {
        jobs[t] = *proto;
        jobs[t].begin = ncells * t / nthreads;
        jobs[t].end = ncells * (t + 1) / nthreads;
        if (pthread_create(&th[t], NULL, fn, &jobs[t]) != 0) { rc = -3; break; }
        started++;
    }
    for (int t = 0; t < started; t++) pthread_join(th[t], NULL);
    if (rc != 0) { /* finish any range a thread could not be started for */
        for (int t = started; t < nthreads; t++) fn(&jobs[t]);
        rc = 0;
    }
    free(jobs);
    free(th);
    return rc;
}

/* S for an arbitrary list of cells (regime m, class k, r index, lam index). */
int kvo_eval_cells(const int32_t* samples, const int64_t* offsets, const int32_t* L, const int32_t* L_in,
                   const int32_t* r, const double* lam, const double* cp, const double* cw, int64_t ncells,
                   const int32_t* cell_m, const int32_t* cell_k, const int32_t* cell_r, const int32_t* cell_l,
                   double* out_S, int nthreads) {
    cells_job p;
    memset(&p, 0, sizeof(p));
    p.samples = samples; p.offsets = offsets; p.L = L; p.L_in = L_in; p.r = r; p.lam = lam;
    p.cp = cp; p.cw = cw; p.cell_m = cell_m; p.cell_k = cell_k; p.cell_r = cell_r; p.cell_l = cell_l;
    p.out = out_S;
    return run_jobs(&p, ncells, nthreads, cells_worker);
}

/* ---- envelope evaluator: the same sum regrouped by affine pieces --------------------------- */

/* C[v] = #{n : x_n <= v}, Sx[v] = sum_{x_n <= v} x_n for v = 0..L (exact integers). */
int kvo_cumulative(const int32_t* x, int64_t n, int32_t L, int64_t* C, int64_t* Sx) {
    if (L < 0) return -1;
    memset(C, 0, sizeof(int64_t) * ((size_t)L + 1));
    memset(Sx, 0, sizeof(int64_t) * ((size_t)L + 1));
    for (int64_t i = 0; i < n; i++) {
        if (x[i] < 0 || x[i] > L) return -1;
        C[x[i]] += 1;
        Sx[x[i]] += x[i];
    }
    for (int32_t v = 1; v <= L; v++) { C[v] += C[v - 1]; Sx[v] += Sx[v - 1]; }
    return 0;
}

static int cmp_double(const void* a, const void* b) {
    double x = *(const double*)a, y = *(const double*)b;
    return (x > y) - (x < y);
}

/* sum_n phi(x_n) for one (eta, lam, c_p, c_w).  phi(x) is the maximum of four
 * affine functions of x: the two branches of Q(eta, x) (c_p (x - eta) and
 * c_w (eta - x); their maximum is Q because c_p, c_w >= 0) and the two moved
 * candidates Q(eta, 0) - lam x and Q(eta, L) - lam (L - x).  Between
 * consecutive pairwise crossings one function is the maximum; the sum over the
 * samples in that piece is alpha * count + beta * sum(x). */
double kvo_envelope_sum(const int64_t* C, const int64_t* Sx, int32_t L, double eta, double lam, double cp,
                        double cw) {
    double alpha[4], beta[4];
    alpha[0] = -cp * eta;                       beta[0] = cp;    /* c_p (x - eta) */
    alpha[1] = cw * eta;                        beta[1] = -cw;   /* c_w (eta - x) */
    alpha[2] = kvo_Q(eta, 0.0, cp, cw);         beta[2] = -lam;  /* Q(eta, 0) - lam x */
    alpha[3] = kvo_Q(eta, (double)L, cp, cw) - lam * (double)L;
    beta[3] = lam;                                               /* Q(eta, L) - lam (L - x) */
    double pts[8];
    int np = 0;
    pts[np++] = 0.0;
    pts[np++] = (double)L;
    for (int i = 0; i < 4; i++)
        for (int j = i + 1; j < 4; j++) {
            if (beta[i] == beta[j]) continue;
            double xc = (alpha[j] - alpha[i]) / (beta[i] - beta[j]);
            if (xc > 0.0 && xc < (double)L) pts[np++] = xc;
        }
    qsort(pts, (size_t)np, sizeof(double), cmp_double);
    double total = 0.0;
    int64_t prev_hi = -1; /* last integer already assigned to a piece */
    for (int t = 0; t + 1 < np; t++) {
        double a = pts[t], b = pts[t + 1];
        if (!(b > a)) continue;
        double mid = 0.5 * (a + b);
        int best = 0;
        double bv = alpha[0] + beta[0] * mid;
        for (int i = 1; i < 4; i++) {
            double v = alpha[i] + beta[i] * mid;
            if (v > bv) { bv = v; best = i; }
        }
        int64_t hi = (t + 2 == np) ? (int64_t)L : (int64_t)floor(b);
        int64_t lo = prev_hi + 1;
        if (hi < lo) continue;
        int64_t cnt = C[hi] - (lo > 0 ? C[lo - 1] : 0);
        int64_t sx = Sx[hi] - (lo > 0 ? Sx[lo - 1] : 0);
        total += alpha[best] * (double)cnt + beta[best] * (double)sx;
        prev_hi = hi;
    }
    return total;
}

typedef struct {
    const int64_t* C;      /* [K][Lmax+1] */
    const int64_t* Sx;
    int64_t stride;        /* Lmax + 1 */
    const int64_t* N;
    const int32_t* L;
    const int32_t* L_in;
    const int32_t* r;
    const double* lam;
    const double* cp;
    const double* cw;
    int32_t K, R, NL;
    double* out;           /* [M][K][R][NL] */
    int64_t begin, end;
} env_job;

static void* env_worker(void* arg) {
    env_job* j = (env_job*)arg;
    for (int64_t c = j->begin; c < j->end; c++) {
        int64_t t = c;
        int l = (int)(t % j->NL); t /= j->NL;
        int ri = (int)(t % j->R); t /= j->R;
        int k = (int)(t % j->K); t /= j->K;
        int m = (int)t;
        double eta = (double)j->r[ri] - (double)j->L_in[k];
        double s = kvo_envelope_sum(j->C + j->stride * k, j->Sx + j->stride * k, j->L[k], eta, j->lam[l],
                                    j->cp[m], j->cw[m]);
        j->out[c] = s / (double)j->N[k];
    }
    return NULL;
}

/* Full S grid [M][K][R][NL] by the envelope evaluator.  C and Sx are [K][stride]. */
int kvo_envelope_grid(const int64_t* C, const int64_t* Sx, int64_t stride, const int64_t* N, const int32_t* L,
                      const int32_t* L_in, const int32_t* r, const double* lam, const double* cp, const double* cw,
                      int32_t M, int32_t K, int32_t R, int32_t NL, double* out_S, int nthreads) {
    int64_t ncells = (int64_t)M * K * R * NL;
    if (nthreads < 1) nthreads = 1;
    if ((int64_t)nthreads > ncells) nthreads = ncells > 0 ? (int)ncells : 1;
    env_job* jobs = (env_job*)malloc(sizeof(env_job) * (size_t)nthreads);
    pthread_t* th = (pthread_t*)malloc(sizeof(pthread_t) * (size_t)nthreads);
    if (!jobs || !th) { free(jobs); free(th); return -2; }
    int started = 0;
    for (int t = 0; t < nthreads; t++) {
        env_job* j = &jobs[t];
        j->C = C; j->Sx = Sx; j->stride = stride; j->N = N; j->L = L; j->L_in = L_in; j->r = r; j->lam = lam;
        j->cp = cp; j->cw = cw; j->K = K; j->R = R; j->NL = NL; j->out = out_S;
        j->begin = ncells * t / nthreads;
        j->end = ncells * (t + 1) / nthreads;
        if (pthread_create(&th[t], NULL, env_worker, j) != 0) break;
        started++;
    }
    for (int t = 0; t < started; t++) pthread_join(th[t], NULL);
    for (int t = started; t < nthreads; t++) env_worker(&jobs[t]);
    free(jobs);
    free(th);
    return 0;
}

/* ---- the exact dual: min over gamma >= 0 of gamma eps + S(eta, gamma) --------------------------- */

/* App. A eq. app_kantorovich without a grid.  g(gamma) is convex and piecewise linear (each sample's
 * phi is a maximum of three lines in gamma: Q(eta,0) - gamma x, Q(eta,x), Q(eta,L) - gamma (L - x)),
 * so its minimum over gamma >= 0 is at gamma = 0 or at a pairwise crossing of one sample's lines.
 * Every candidate is evaluated with the envelope sum; the smallest value (first in candidate order on
 * ties) is returned with its gamma.  `vals` holds the class's distinct sample values. */
void kvo_exact_dual(const int64_t* C, const int64_t* Sx, int32_t L, int64_t N, const int32_t* vals, int64_t nvals,
                    double eta, double eps, double cp, double cw, double* out_cost, double* out_gamma) {
    const double q0 = kvo_Q(eta, 0.0, cp, cw), qL = kvo_Q(eta, (double)L, cp, cw);
    double best = kvo_envelope_sum(C, Sx, L, eta, 0.0, cp, cw) / (double)N;  /* gamma = 0 */
    double bg = 0.0;
    for (int64_t i = 0; i < nvals; i++) {
        const double x = (double)vals[i], qx = kvo_Q(eta, x, cp, cw);
        double cand[3];
        int nc = 0;
        if (x > 0.0) cand[nc++] = (q0 - qx) / x;                       /* Q(0) - g x = Q(x)      */
        if (x < (double)L) cand[nc++] = (qL - qx) / ((double)L - x);   /* Q(L) - g (L-x) = Q(x)  */
        if (2.0 * x != (double)L) cand[nc++] = (q0 - qL) / (2.0 * x - (double)L); /* the two moved */
        for (int c = 0; c < nc; c++) {
            const double g = cand[c];
            if (!(g > 0.0) || !isfinite(g)) continue;
            const double v = g * eps + kvo_envelope_sum(C, Sx, L, eta, g, cp, cw) / (double)N;
            if (v < best) { best = v; bg = g; }
        }
    }
    *out_cost = best;
    *out_gamma = bg;
}

typedef struct {
    const int64_t* C;
    const int64_t* Sx;
    int64_t stride;
    const int64_t* N;
    const int32_t* L;
    const int32_t* L_in;
    const int32_t* vals;     /* distinct values, class k at vals_off[k] */
    const int64_t* vals_off;
    const int32_t* r;
    const double* eps;
    const double* cp;
    const double* cw;
    int32_t K, R, E;
    double* cost;            /* [M][E][K][R] */
    double* gamma;
    int64_t begin, end;
} dual_job;

static void* dual_worker(void* arg) {
    dual_job* j = (dual_job*)arg;
    for (int64_t c = j->begin; c < j->end; c++) {
        int64_t t = c;
        const int ri = (int)(t % j->R); t /= j->R;
        const int k = (int)(t % j->K); t /= j->K;
        const int e = (int)(t % j->E);
        const int m = (int)(t / j->E);
        kvo_exact_dual(j->C + j->stride * k, j->Sx + j->stride * k, j->L[k], j->N[k], j->vals + j->vals_off[k],
                       j->vals_off[k + 1] - j->vals_off[k], (double)j->r[ri] - (double)j->L_in[k], j->eps[e],
                       j->cp[m], j->cw[m], &j->cost[c], &j->gamma[c]);
    }
    return NULL;
}

int kvo_exact_dual_grid(const int64_t* C, const int64_t* Sx, int64_t stride, const int64_t* N, const int32_t* L,
                        const int32_t* L_in, const int32_t* vals, const int64_t* vals_off, const int32_t* r,
                        const double* eps, const double* cp, const double* cw, int32_t M, int32_t E, int32_t K,
                        int32_t R, double* cost, double* gamma, int nthreads) {
    const int64_t ncells = (int64_t)M * E * K * R;
    if (nthreads < 1) nthreads = 1;
    if ((int64_t)nthreads > ncells) nthreads = ncells > 0 ? (int)ncells : 1;
    dual_job* jobs = (dual_job*)malloc(sizeof(dual_job) * (size_t)nthreads);
    pthread_t* th = (pthread_t*)malloc(sizeof(pthread_t) * (size_t)nthreads);
    if (!jobs || !th) { free(jobs); free(th); return -2; }
    int started = 0;
    for (int t = 0; t < nthreads; t++) {
        dual_job* j = &jobs[t];
        j->C = C; j->Sx = Sx; j->stride = stride; j->N = N; j->L = L; j->L_in = L_in; j->vals = vals;
        j->vals_off = vals_off; j->r = r; j->eps = eps; j->cp = cp; j->cw = cw; j->K = K; j->R = R; j->E = E;
        j->cost = cost; j->gamma = gamma;
        j->begin = ncells * t / nthreads;
        j->end = ncells * (t + 1) / nthreads;
        if (pthread_create(&th[t], NULL, dual_worker, j) != 0) break;
        started++;
    }
    for (int t = 0; t < started; t++) pthread_join(th[t], NULL);
    for (int t = started; t < nthreads; t++) dual_worker(&jobs[t]);
    free(jobs);
    free(th);
    return 0;
}
