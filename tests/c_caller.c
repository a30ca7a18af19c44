/*
 * A plain C11 caller of libgnmr, test infrastructure for
 * tests/test_gpu_c_caller.py: no Python and no torch in the process.
 *
 * Reads a layout and a sequence of fp32 step arenas from a binary file,
 * creates a handle, runs one gnmr_step per arena on a stream of its own,
 * copies the mask and every statistic back and prints them as text.
 *
 * Input (little-endian): int64 U, n (arena elements), steps, window, max_o,
 * lock_len; double alpha, beta, eps; int64 offsets[U], lengths[U]; then
 * float arena[steps][n].
 * Output: per step one line "step t counts c0 c1", then U lines
 * "b mask lock norm gnmr dgnmr risk" (doubles printed exactly, %a).
 * Exit status 0 on success; any failed call prints its reason and exits 1.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <cuda_runtime.h>

#include "gnmr.h"

#define CUDA_OK(x)                                                                        \
    do {                                                                                  \
        cudaError_t e_ = (x);                                                             \
        if (e_ != cudaSuccess) {                                                          \
            fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));                      \
            exit(1);                                                                      \
        }                                                                                 \
    } while (0)

#define GNMR_OK_OR_DIE(h, x)                                                              \
    do {                                                                                  \
        gnmr_status s_ = (x);                                                             \
        if (s_ != GNMR_OK) {                                                              \
            fprintf(stderr, "%s: %s (%s)\n", #x, gnmr_status_string(s_), gnmr_last_error(h)); \
            exit(1);                                                                      \
        }                                                                                 \
    } while (0)

static void read_all(FILE *f, void *dst, size_t bytes)
{
    if (fread(dst, 1, bytes, f) != bytes) {
        fprintf(stderr, "input file too short\n");
        exit(1);
    }
}

static void *host_alloc(size_t bytes)
{
    void *p = malloc(bytes ? bytes : 1);
    if (!p) {
        fprintf(stderr, "out of host memory\n");
        exit(1);
    }
    return p;
}

int main(int argc, char **argv)
{
    if (argc != 2) {
        fprintf(stderr, "usage: %s <input file>\n", argv[0]);
        return 1;
    }
    FILE *f = fopen(argv[1], "rb");
    if (!f) {
        perror(argv[1]);
        return 1;
    }
    int64_t hdr[6];
    double thr[3];
    read_all(f, hdr, sizeof hdr);
    read_all(f, thr, sizeof thr);
    const int64_t U = hdr[0], n = hdr[1], steps = hdr[2];
    if (U < 1 || U > (1 << 24) || n < 1 || steps < 1) {
        fprintf(stderr, "bad header\n");
        return 1;
    }
    int64_t *off = host_alloc(sizeof(int64_t) * U);
    int64_t *len = host_alloc(sizeof(int64_t) * U);
    read_all(f, off, sizeof(int64_t) * U);
    read_all(f, len, sizeof(int64_t) * U);

    gnmr_config cfg;
    gnmr_config_defaults(&cfg);
    cfg.num_units = (int32_t)U;
    cfg.offsets = off;
    cfg.lengths = len;
    cfg.dtype = GNMR_DTYPE_F32;
    cfg.window = (int32_t)hdr[3];
    cfg.max_o = (int32_t)hdr[4];
    cfg.lock_len = (int32_t)hdr[5];
    cfg.alpha_init = cfg.alpha_main = thr[0];
    cfg.beta_init = cfg.beta_main = thr[1];
    cfg.eps = thr[2];
    gnmr_handle *h = NULL;
    GNMR_OK_OR_DIE(NULL, gnmr_create(&cfg, &h));

    float *arena_h = host_alloc(sizeof(float) * n);
    void *arena_d = NULL;
    uint8_t *mask_d = NULL;
    double *stat_d = NULL;
    int32_t *lock_d = NULL, *counts_d = NULL;
    CUDA_OK(cudaMalloc(&arena_d, sizeof(float) * n));
    CUDA_OK(cudaMalloc((void **)&mask_d, U));
    CUDA_OK(cudaMalloc((void **)&stat_d, sizeof(double) * 4 * U));
    CUDA_OK(cudaMalloc((void **)&lock_d, sizeof(int32_t) * U));
    CUDA_OK(cudaMalloc((void **)&counts_d, sizeof(int32_t) * 2));
    cudaStream_t stream;
    CUDA_OK(cudaStreamCreate(&stream));

    gnmr_stats stats = {0};
    stats.norm = stat_d;
    stats.gnmr = stat_d + U;
    stats.dgnmr = stat_d + 2 * U;
    stats.risk = stat_d + 3 * U;
    stats.lock = lock_d;
    stats.counts = counts_d;

    uint8_t *mask_h = host_alloc(U);
    double *stat_h = host_alloc(sizeof(double) * 4 * U);
    int32_t *lock_h = host_alloc(sizeof(int32_t) * U);
    int32_t counts_h[2];
    for (int64_t t = 0; t < steps; ++t) {
        read_all(f, arena_h, sizeof(float) * n);
        CUDA_OK(cudaMemcpyAsync(arena_d, arena_h, sizeof(float) * n, cudaMemcpyHostToDevice, stream));
        GNMR_OK_OR_DIE(h, gnmr_step(h, arena_d, n, (void *)stream, mask_d, &stats));
        CUDA_OK(cudaMemcpyAsync(mask_h, mask_d, U, cudaMemcpyDeviceToHost, stream));
        CUDA_OK(cudaMemcpyAsync(stat_h, stat_d, sizeof(double) * 4 * U, cudaMemcpyDeviceToHost, stream));
        CUDA_OK(cudaMemcpyAsync(lock_h, lock_d, sizeof(int32_t) * U, cudaMemcpyDeviceToHost, stream));
        CUDA_OK(cudaMemcpyAsync(counts_h, counts_d, sizeof counts_h, cudaMemcpyDeviceToHost, stream));
        CUDA_OK(cudaStreamSynchronize(stream));
        printf("step %lld counts %d %d\n", (long long)(t + 1), counts_h[0], counts_h[1]);
        for (int64_t b = 0; b < U; ++b)
            printf("%lld %d %d %a %a %a %a\n", (long long)b, mask_h[b], lock_h[b], stat_h[b], stat_h[U + b],
                   stat_h[2 * U + b], stat_h[3 * U + b]);
    }
    fclose(f);
    GNMR_OK_OR_DIE(h, gnmr_destroy(h));
    CUDA_OK(cudaStreamDestroy(stream));
    CUDA_OK(cudaFree(arena_d));
    CUDA_OK(cudaFree(mask_d));
    CUDA_OK(cudaFree(stat_d));
    CUDA_OK(cudaFree(lock_d));
    CUDA_OK(cudaFree(counts_d));
    free(off);
    free(len);
    free(arena_h);
    free(mask_h);
    free(stat_h);
    free(lock_h);
    return 0;
}
