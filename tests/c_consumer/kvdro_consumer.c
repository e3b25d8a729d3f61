/*
 * A plain C caller of the library, for the tests: it includes only kvdro.h, passes host buffers
 * only (no CUDA header and no device memory of its own), reads a workload as whitespace-separated
 * text on stdin and prints every output as text.  tests/test_c_consumer.py builds it with gcc
 * against libkvdro.so and checks what it prints against the oracle.
 *
 * Input:  K, offsets[K+1], lengths[offsets[K]], L_max[K], L_in[K], R, r[R], NL, lam[NL], E,
 *         eps[E], M, c_p[M], c_w[M], F, fractiles[F], precision (a kvdro_precision value).
 * Output: one line per array, "<name> <count> <values...>", FP values with 17 significant digits.
 *         On an error: "error <status> <message>" and exit status 1.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include "kvdro.h"

static void* take(size_t n, size_t size) {
    void* p = calloc(n ? n : 1, size);
    if (!p) {
        fprintf(stderr, "out of host memory\n");
        exit(2);
    }
    return p;
}

static int64_t read_i64(void) {
    long long v;
    if (scanf("%lld", &v) != 1) {
        fprintf(stderr, "bad input\n");
        exit(2);
    }
    return (int64_t)v;
}

static double read_f64(void) {
    double v;
    if (scanf("%lf", &v) != 1) {
        fprintf(stderr, "bad input\n");
        exit(2);
    }
    return v;
}

static void put_i32(const char* name, const int32_t* v, int64_t n) {
    printf("%s %lld", name, (long long)n);
    for (int64_t i = 0; i < n; i++) printf(" %d", v[i]);
    printf("\n");
}

static void put_f64(const char* name, const double* v, int64_t n) {
    printf("%s %lld", name, (long long)n);
    for (int64_t i = 0; i < n; i++) printf(" %.17g", v[i]);
    printf("\n");
}

static int check(kvdro_ctx* ctx, int status) {
    if (status != KVDRO_OK) {
        printf("error %d %s\n", status, kvdro_last_error(ctx));
        kvdro_destroy(ctx);
        exit(1);
    }
    return status;
}

int main(void) {
    const int32_t K = (int32_t)read_i64();
    int64_t* offsets = take((size_t)K + 1, sizeof(int64_t));
    for (int32_t k = 0; k <= K; k++) offsets[k] = read_i64();
    const int64_t total = offsets[K];
    int32_t* lengths = take((size_t)total, sizeof(int32_t));
    for (int64_t i = 0; i < total; i++) lengths[i] = (int32_t)read_i64();
    int32_t* L_max = take((size_t)K, sizeof(int32_t));
    int32_t* L_in = take((size_t)K, sizeof(int32_t));
    for (int32_t k = 0; k < K; k++) L_max[k] = (int32_t)read_i64();
    for (int32_t k = 0; k < K; k++) L_in[k] = (int32_t)read_i64();
    const int32_t R = (int32_t)read_i64();
    int32_t* r = take((size_t)R, sizeof(int32_t));
    for (int32_t i = 0; i < R; i++) r[i] = (int32_t)read_i64();
    const int32_t NL = (int32_t)read_i64();
    double* lam = take((size_t)NL, sizeof(double));
    for (int32_t i = 0; i < NL; i++) lam[i] = read_f64();
    const int32_t E = (int32_t)read_i64();
    double* eps = take((size_t)E, sizeof(double));
    for (int32_t i = 0; i < E; i++) eps[i] = read_f64();
    const int32_t M = (int32_t)read_i64();
    double* c_p = take((size_t)M, sizeof(double));
    double* c_w = take((size_t)M, sizeof(double));
    for (int32_t i = 0; i < M; i++) c_p[i] = read_f64();
    for (int32_t i = 0; i < M; i++) c_w[i] = read_f64();
    const int32_t F = (int32_t)read_i64();
    double* fractiles = take((size_t)F, sizeof(double));
    for (int32_t i = 0; i < F; i++) fractiles[i] = read_f64();
    const int precision = (int)read_i64();
    if (precision != KVDRO_FP64 && precision != KVDRO_EXACT && precision != KVDRO_ENVELOPE) {
        fprintf(stderr, "this caller reads FP64 outputs: precision must be FP64, EXACT or ENVELOPE\n");
        return 2;
    }

    const int64_t rows = (int64_t)M * E * K, cells = rows * R;
    int32_t* quant = take((size_t)K * F, sizeof(int32_t));
    double* cost = take((size_t)cells, sizeof(double));
    int32_t* lam_idx = take((size_t)cells, sizeof(int32_t));
    int32_t* r_idx = take((size_t)rows, sizeof(int32_t));
    double* min_cost = take((size_t)rows, sizeof(double));
    double* fhat = take((size_t)rows, sizeof(double));
    int32_t* sorted = take((size_t)total, sizeof(int32_t));

    kvdro_ctx* ctx = NULL;
    check(NULL, kvdro_create(&ctx, 0));
    check(ctx, kvdro_load_samples(ctx, K, offsets, lengths, L_max, L_in, NULL));
    check(ctx, kvdro_quantiles(ctx, F, fractiles, quant, NULL));
    check(ctx, kvdro_sorted_samples(ctx, sorted, NULL));
    check(ctx, kvdro_eval_grid(ctx, precision, R, r, NL, lam, E, eps, M, c_p, c_w, NULL, cost, lam_idx, r_idx,
                               min_cost, fhat, NULL));
    check(ctx, kvdro_sync(ctx));
    kvdro_destroy(ctx);

    put_i32("quant", quant, (int64_t)K * F);
    put_i32("sorted", sorted, total);
    put_f64("cost", cost, cells);
    put_i32("lam_idx", lam_idx, cells);
    put_i32("r_idx", r_idx, rows);
    put_f64("min_cost", min_cost, rows);
    put_f64("fhat", fhat, rows);
    return 0;
}
