/*
 * A plain C client of libcpdp's C ABI (include/cpdp.h): no Python, no torch.
 * Reads a problem from stdin, runs it through cpdp_step, and prints the state
 * after every step, so a test can compare it with expected values. With the
 * argument "host", the gradients stay in page-locked host memory and go
 * through cpdp_bind_staging / cpdp_step_host instead. With "staged" or
 * "shuffle", the reconcile runs its shared-memory-staged variant
 * (cpdp_set_reconcile_staging) or its warp-shuffle variant
 * (cpdp_set_reconcile_shuffle).
 *
 * Input (whitespace separated):
 *   W N K T lr momentum weight_decay beta alpha
 *   theta0[N]
 *   T times: grads[W][N]
 * Output per step t: "t sync" then the rows of params, mom, then anchor, slow_v
 * (one line each, values printed with %.9g, enough to round-trip a float).
 * Exit status 0 on success; on a library or CUDA error, prints the message
 * to stderr and exits with status 2.
 */
#include <cuda_runtime.h>
#include <stdio.h>
#include <stdlib.h>

#include "cpdp.h"

#define CUDA_OK(x)                                                               \
    do {                                                                         \
        cudaError_t e_ = (x);                                                    \
        if (e_ != cudaSuccess) {                                                 \
            fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));             \
            exit(2);                                                             \
        }                                                                        \
    } while (0)

#define CPDP_OK_OR_DIE(ctx, x)                                                   \
    do {                                                                         \
        cpdp_status s_ = (x);                                                    \
        if (s_ != CPDP_OK) {                                                     \
            fprintf(stderr, "%s -> %d: %s\n", #x, (int)s_, cpdp_last_error(ctx)); \
            exit(2);                                                             \
        }                                                                        \
    } while (0)

static void print_rows(const float *dev, int rows, long long n) {
    float *h = (float *)malloc((size_t)rows * (size_t)n * sizeof(float));
    CUDA_OK(cudaMemcpy(h, dev, (size_t)rows * (size_t)n * sizeof(float), cudaMemcpyDeviceToHost));
    for (int i = 0; i < rows; ++i) {
        for (long long j = 0; j < n; ++j) printf(j ? " %.9g" : "%.9g", h[(size_t)i * (size_t)n + (size_t)j]);
        printf("\n");
    }
    free(h);
}

int main(int argc, char **argv) {
    const char mode = argc > 1 ? argv[1][0] : 'd';
    const int from_host = mode == 'h';
    int W, K, T;
    long long N;
    float lr, mu, wd, beta, alpha;
    if (scanf("%d %lld %d %d %f %f %f %f %f", &W, &N, &K, &T, &lr, &mu, &wd, &beta, &alpha) != 9) return 1;
    float *theta0 = (float *)malloc((size_t)N * sizeof(float));
    float *grads = (float *)malloc((size_t)T * (size_t)W * (size_t)N * sizeof(float));
    for (long long j = 0; j < N; ++j)
        if (scanf("%f", &theta0[j]) != 1) return 1;
    for (long long k = 0; k < (long long)T * W * N; ++k)
        if (scanf("%f", &grads[k]) != 1) return 1;

    float *d_params, *d_mom, *d_anchor, *d_v, *d_theta0, *d_grads, *d_stage1, *h_grads = NULL;
    const size_t state = (size_t)W * (size_t)N * sizeof(float), row = (size_t)N * sizeof(float);
    CUDA_OK(cudaMalloc((void **)&d_params, state));
    CUDA_OK(cudaMalloc((void **)&d_mom, state));
    CUDA_OK(cudaMalloc((void **)&d_anchor, row));
    CUDA_OK(cudaMalloc((void **)&d_v, row));
    CUDA_OK(cudaMalloc((void **)&d_theta0, row));
    CUDA_OK(cudaMalloc((void **)&d_grads, state));
    CUDA_OK(cudaMalloc((void **)&d_stage1, state));
    if (from_host) CUDA_OK(cudaHostAlloc((void **)&h_grads, (size_t)T * state, cudaHostAllocDefault));
    CUDA_OK(cudaMemcpy(d_theta0, theta0, row, cudaMemcpyHostToDevice));

    cpdp_ctx *ctx = NULL;
    CPDP_OK_OR_DIE(NULL, cpdp_create(&ctx, W, N, NULL, 0, lr, mu, wd, K, beta, alpha));
    CPDP_OK_OR_DIE(ctx, cpdp_bind(ctx, d_params, d_mom, d_anchor, d_v));
    CPDP_OK_OR_DIE(ctx, cpdp_init_params(ctx, d_theta0, NULL));
    if (mode == 's' && argv[1][1] == 't') CPDP_OK_OR_DIE(ctx, cpdp_set_reconcile_staging(ctx, 2));
    if (mode == 's' && argv[1][1] == 'h') CPDP_OK_OR_DIE(ctx, cpdp_set_reconcile_shuffle(ctx, 1));
    if (from_host) {
        for (size_t k = 0; k < (size_t)T * (size_t)W * (size_t)N; ++k) h_grads[k] = grads[k];
        CPDP_OK_OR_DIE(ctx, cpdp_bind_staging(ctx, d_grads, d_stage1, state));
    }
    for (int t = 1; t <= T; ++t) {
        int synced = -1;
        if (from_host) {
            CPDP_OK_OR_DIE(ctx, cpdp_step_host(ctx, h_grads + (size_t)(t - 1) * (size_t)W * (size_t)N, CPDP_F32, t, T,
                                               NULL, &synced));
        } else {
            CUDA_OK(cudaMemcpy(d_grads, grads + (size_t)(t - 1) * (size_t)W * (size_t)N, state, cudaMemcpyHostToDevice));
            CPDP_OK_OR_DIE(ctx, cpdp_step(ctx, d_grads, CPDP_F32, t, T, NULL, &synced));
        }
        CUDA_OK(cudaDeviceSynchronize());
        printf("%d %d\n", t, synced);
        print_rows(d_params, W, N);
        print_rows(d_mom, W, N);
        print_rows(d_anchor, 1, N);
        print_rows(d_v, 1, N);
    }
    const char *kernel = NULL;
    CPDP_OK_OR_DIE(ctx, cpdp_reconcile_kernel(ctx, &kernel));
    printf("kernel %s\n", kernel);
    CPDP_OK_OR_DIE(NULL, cpdp_destroy(ctx));
    cudaFree(d_params);
    cudaFree(d_mom);
    cudaFree(d_anchor);
    cudaFree(d_v);
    cudaFree(d_theta0);
    cudaFree(d_grads);
    cudaFree(d_stage1);
    if (h_grads != NULL) cudaFreeHost(h_grads);
    free(theta0);
    free(grads);
    return 0;
}
