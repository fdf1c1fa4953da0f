/* A RelaySGD run driven from C through the library's ABI alone (no Python):
 * the sequence a C caller writes.  Used by tests/test_gpu_c_abi.py, which
 * compares the models it writes with the Python binding's run of the same
 * configuration.
 *
 * usage: c_abi_run <tree: chain|binary> <n> <d> <steps> <mode> <out.bin> [fused|host]
 * writes x (float32 [n][d]) and the two metrics (double [2]) to out.bin; with
 * "fused" the steps run as one relay_steps call instead of relay_step calls;
 * with "host" the state lives in page-locked host memory and every step is a
 * relay_step_host call (centres regenerated, chunks of 1024 coordinates). */
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "relaysum.h"

#define CHECK(call)                                                                   \
    do {                                                                              \
        int rc_ = (call);                                                             \
        if (rc_ != RELAY_OK) {                                                        \
            fprintf(stderr, "%s failed: %s\n", #call, relay_error_string(rc_));      \
            return 1;                                                                 \
        }                                                                             \
    } while (0)

#define CUDA(call)                                                                    \
    do {                                                                              \
        cudaError_t e_ = (call);                                                      \
        if (e_ != cudaSuccess) {                                                      \
            fprintf(stderr, "%s failed: %s\n", #call, cudaGetErrorString(e_));       \
            return 1;                                                                 \
        }                                                                             \
    } while (0)

int main(int argc, char **argv) {
    if (argc != 7 && !(argc == 8 && (strcmp(argv[7], "fused") == 0 || strcmp(argv[7], "host") == 0))) {
        fprintf(stderr, "usage: %s chain|binary n d steps mode out.bin [fused|host]\n", argv[0]);
        return 2;
    }
    const int fused = argc == 8 && strcmp(argv[7], "fused") == 0;
    const int host = argc == 8 && strcmp(argv[7], "host") == 0;
    const int binary = strcmp(argv[1], "binary") == 0;
    const int n = atoi(argv[2]);
    const int64_t d = atoll(argv[3]);
    const int64_t steps = atoll(argv[4]);
    const int mode = atoi(argv[5]);
    if (n < 2 || n > RELAY_MAX_N || d < 1 || steps < 0) return 2;

    /* the tree: a chain i - i+1, or the heap binary tree parent(i) = (i-1)/2 */
    int32_t *edges = (int32_t *)malloc(sizeof(int32_t) * 2 * (size_t)(n - 1));
    for (int i = 1; i < n; ++i) {
        edges[2 * (i - 1)] = binary ? (i - 1) / 2 : i - 1;
        edges[2 * (i - 1) + 1] = i;
    }
    relay_handle *h = NULL;
    CHECK(relay_create(&h, n, d, edges, n - 1));
    free(edges);
    CHECK(relay_set_rebuild_mode(h, mode));
    const int64_t ld = relay_ld(h);
    const int E = relay_num_edges(h);

    float *x, *mu, *msg[2], *mix;
    int32_t *counts;
    double *out;
    CUDA(cudaMalloc((void **)&x, sizeof(float) * (size_t)n * (size_t)ld));
    CUDA(cudaMalloc((void **)&mu, sizeof(float) * (size_t)n * (size_t)ld));
    CUDA(cudaMalloc((void **)&msg[0], sizeof(float) * (size_t)E * (size_t)ld));
    CUDA(cudaMalloc((void **)&msg[1], sizeof(float) * (size_t)E * (size_t)ld));
    CUDA(cudaMalloc((void **)&counts, sizeof(int32_t) * (size_t)E));
    CUDA(cudaMalloc((void **)&out, sizeof(double) * 2));
    /* one Gaussian centre per worker: the identity mixture */
    float *mix_h = (float *)calloc((size_t)n * (size_t)n, sizeof(float));
    for (int i = 0; i < n; ++i) mix_h[(size_t)i * n + i] = 1.0f;
    CUDA(cudaMalloc((void **)&mix, sizeof(float) * (size_t)n * (size_t)n));
    CUDA(cudaMemcpy(mix, mix_h, sizeof(float) * (size_t)n * (size_t)n, cudaMemcpyHostToDevice));

    cudaStream_t stream;
    CUDA(cudaStreamCreate(&stream));
    relay_stream_t s = (relay_stream_t)stream;
    const float lr = 0.1f, sigma = 0.1f;
    const uint64_t seed = 0, mu_seed = 0;
    if (host) {
        CHECK(relay_set_objective_generated(h, mix_h, n, 2.0f, mu_seed, sigma));
    } else {
        CHECK(relay_fill_objective(h, mu, mix, n, 2.0f, mu_seed, s));
        CHECK(relay_set_objective(h, mu, sigma));
    }
    free(mix_h);
    CHECK(relay_init(h, x, msg[0], msg[1], counts, 0.0f, seed, s));
    if (host) {
        /* the state moves to page-locked host memory; the device keeps only
         * the plan's staging (three sets of one chunk) */
        float *x_p, *m_p[2];
        int32_t *c_p;
        const size_t xb = sizeof(float) * (size_t)n * (size_t)ld, mb = sizeof(float) * (size_t)E * (size_t)ld;
        CUDA(cudaMallocHost((void **)&x_p, xb));
        CUDA(cudaMallocHost((void **)&m_p[0], mb));
        CUDA(cudaMallocHost((void **)&m_p[1], mb));
        CUDA(cudaMallocHost((void **)&c_p, sizeof(int32_t) * (size_t)E));
        CUDA(cudaMemcpyAsync(x_p, x, xb, cudaMemcpyDeviceToHost, stream));
        CUDA(cudaMemcpyAsync(m_p[0], msg[0], mb, cudaMemcpyDeviceToHost, stream));
        CUDA(cudaMemcpyAsync(c_p, counts, sizeof(int32_t) * (size_t)E, cudaMemcpyDeviceToHost, stream));
        const int64_t staging_bytes = relay_host_staging_bytes(h, 1024, 3);
        if (staging_bytes < 0) return 1;
        void *staging;
        CUDA(cudaMalloc(&staging, (size_t)staging_bytes));
        relay_host_plan *plan = NULL;
        CHECK(relay_host_plan_create(&plan, h, 1024, 3, staging, staging_bytes, 0));
        for (int64_t t = 0; t < steps; ++t)
            CHECK(relay_step_host(plan, x_p, m_p[t & 1], m_p[(t + 1) & 1], c_p, lr, seed, t, s));
        CUDA(cudaMemcpyAsync(x, x_p, xb, cudaMemcpyHostToDevice, stream));
        CUDA(cudaStreamSynchronize(stream));
        relay_host_plan_destroy(plan);
        cudaFree(staging);
        cudaFreeHost(x_p);
        cudaFreeHost(m_p[0]);
        cudaFreeHost(m_p[1]);
        cudaFreeHost(c_p);
    } else if (fused) {
        CHECK(relay_steps(h, x, msg[0], msg[1], counts, lr, seed, 0, steps, s));
    } else {
        for (int64_t t = 0; t < steps; ++t)
            CHECK(relay_step(h, x, msg[t & 1], msg[(t + 1) & 1], counts, lr, seed, t, s));
    }
    CHECK(relay_metrics_static(h, x, out, s));
    CUDA(cudaStreamSynchronize(stream));

    float *x_h = (float *)malloc(sizeof(float) * (size_t)n * (size_t)d);
    CUDA(cudaMemcpy2D(x_h, sizeof(float) * (size_t)d, x, sizeof(float) * (size_t)ld, sizeof(float) * (size_t)d,
                      (size_t)n, cudaMemcpyDeviceToHost));
    double m[2];
    CUDA(cudaMemcpy(m, out, sizeof(m), cudaMemcpyDeviceToHost));
    FILE *f = fopen(argv[6], "wb");
    if (!f) return 1;
    fwrite(x_h, sizeof(float), (size_t)n * (size_t)d, f);
    fwrite(m, sizeof(double), 2, f);
    fclose(f);
    free(x_h);

    cudaFree(x);
    cudaFree(mu);
    cudaFree(msg[0]);
    cudaFree(msg[1]);
    cudaFree(counts);
    cudaFree(out);
    cudaFree(mix);
    cudaStreamDestroy(stream);
    relay_destroy(h);
    return 0;
}
