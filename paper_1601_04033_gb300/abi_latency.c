/*
 * abi_latency -- times small dense server passes from C through the ABI of
 * include/fasgd.h, to split the cost of one push + apply step into
 *   host:  the ABI calls themselves (fasgd_push x K, fasgd_apply_pending),
 *          measured on the host clock while the GPU runs behind;
 *   issue: the GPU-side time per step of an eager loop (CUDA events around
 *          the loop on the handle's stream): the kernel plus any idle time
 *          the host leaves between launches;
 *   graph: the GPU-side time per step of the same steps captured once in a
 *          CUDA graph and replayed, with no host work between the kernels.
 * The Python binding adds its own (ctypes) cost on top of "host"; bench.py
 * reports that figure for the same workloads.
 *
 * Every step applies K pushes at the current timestamp (tau = 0) with
 * gradients from a pool of 2K device vectors; the arithmetic of the pass
 * does not depend on the values, only the sizes matter for timing.
 *
 * usage: abi_latency P K steps [variant]    (variant: 0 ASGD .. 3 FASGD_STD)
 * prints one JSON line.
 */
#define _POSIX_C_SOURCE 199309L
#include <stdio.h>
#include <stdlib.h>
#include <time.h>

#include <cuda_runtime_api.h>

#include "fasgd.h"

#define CHECK_CUDA(x)                                                             \
    do {                                                                          \
        cudaError_t st_ = (x);                                                    \
        if (st_ != cudaSuccess) {                                                 \
            fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(st_));             \
            return 2;                                                             \
        }                                                                         \
    } while (0)

#define CHECK_ABI(h, x)                                                           \
    do {                                                                          \
        int rc_ = (x);                                                            \
        if (rc_ != FASGD_OK) {                                                    \
            fprintf(stderr, "%s: %d %s\n", #x, rc_, fasgd_last_error(h));         \
            return 3;                                                             \
        }                                                                         \
    } while (0)

static double now_us(void) {
    struct timespec ts;
    clock_gettime(CLOCK_MONOTONIC, &ts);
    return ts.tv_sec * 1e6 + ts.tv_nsec * 1e-3;
}

/* One step: K pushes at the current timestamp, then one apply of K. */
static int step(fasgd_t* h, int K, int lambda, float* const* pool, int R, long s) {
    const int64_t T = fasgd_timestamp(h);
    for (int k = 0; k < K; ++k) {
        const int rc = fasgd_push(h, (int32_t)((s * K + k) % lambda), T, pool[(s * K + k) % R]);
        if (rc != FASGD_OK) return rc;
    }
    return fasgd_apply_pending(h, K);
}

int main(int argc, char** argv) {
    if (argc < 4) {
        fprintf(stderr, "usage: %s P K steps [variant]\n", argv[0]);
        return 1;
    }
    const int64_t P = atoll(argv[1]);
    const int K = atoi(argv[2]);
    const long steps = atol(argv[3]);
    const int variant = argc > 4 ? atoi(argv[4]) : FASGD_FASGD;
    const int lambda = 32, R = 2 * K, warm = 100;
    if (P < 1 || K < 1 || K > FASGD_KMAX || steps < 1) return 1;

    cudaStream_t stream;
    CHECK_CUDA(cudaSetDevice(0));
    CHECK_CUDA(cudaStreamCreateWithFlags(&stream, cudaStreamNonBlocking));
    float* pool[2 * FASGD_KMAX];
    const size_t bytes = (size_t)((P + 3) / 4 * 4) * sizeof(float);
    for (int r = 0; r < R; ++r) {
        CHECK_CUDA(cudaMalloc((void**)&pool[r], bytes));
        CHECK_CUDA(cudaMemset(pool[r], 0x3b + r % 4, bytes));   /* small positive floats */
    }
    fasgd_t* h = NULL;
    CHECK_ABI(NULL, fasgd_create(&h, P, lambda, 0.001f, variant));
    CHECK_ABI(h, fasgd_set_stream(h, stream));

    for (long s = 0; s < warm; ++s) CHECK_ABI(h, step(h, K, lambda, pool, R, s));
    CHECK_CUDA(cudaStreamSynchronize(stream));

    /* Eager loop: host time of the calls, GPU time between events. */
    cudaEvent_t e0, e1;
    CHECK_CUDA(cudaEventCreate(&e0));
    CHECK_CUDA(cudaEventCreate(&e1));
    CHECK_CUDA(cudaEventRecord(e0, stream));
    const double t0 = now_us();
    for (long s = 0; s < steps; ++s) CHECK_ABI(h, step(h, K, lambda, pool, R, s));
    const double t1 = now_us();
    CHECK_CUDA(cudaEventRecord(e1, stream));
    CHECK_CUDA(cudaStreamSynchronize(stream));
    const double t2 = now_us();
    float eager_ms = 0.f;
    CHECK_CUDA(cudaEventElapsedTime(&eager_ms, e0, e1));

    /* The same steps captured in one graph and replayed. */
    const long gsteps = steps < 200 ? steps : 200;
    const int reps = 10;
    cudaGraph_t graph;
    cudaGraphExec_t exec;
    CHECK_CUDA(cudaStreamBeginCapture(stream, cudaStreamCaptureModeThreadLocal));
    for (long s = 0; s < gsteps; ++s) {
        const int rc = step(h, K, lambda, pool, R, s);
        if (rc != FASGD_OK) {
            cudaStreamEndCapture(stream, &graph);
            CHECK_ABI(h, rc);
        }
    }
    CHECK_CUDA(cudaStreamEndCapture(stream, &graph));
    CHECK_CUDA(cudaGraphInstantiate(&exec, graph, 0));
    CHECK_CUDA(cudaGraphLaunch(exec, stream));           /* warm-up replay */
    CHECK_CUDA(cudaStreamSynchronize(stream));
    CHECK_CUDA(cudaEventRecord(e0, stream));
    for (int r = 0; r < reps; ++r) CHECK_CUDA(cudaGraphLaunch(exec, stream));
    CHECK_CUDA(cudaEventRecord(e1, stream));
    CHECK_CUDA(cudaStreamSynchronize(stream));
    float graph_ms = 0.f;
    CHECK_CUDA(cudaEventElapsedTime(&graph_ms, e0, e1));
    CHECK_ABI(h, fasgd_sync(h));

    const double host_us = (t1 - t0) / steps;
    printf("{\"P\": %lld, \"K\": %d, \"variant\": %d, \"steps\": %ld, "
           "\"host_us_per_step\": %.3f, \"wall_us_per_step\": %.3f, "
           "\"eager_gpu_us_per_step\": %.3f, \"graph_gpu_us_per_step\": %.3f, "
           "\"graph_steps\": %ld, \"graph_replays\": %d}\n",
           (long long)P, K, variant, steps, host_us, (t2 - t0) / steps,
           eager_ms * 1e3 / steps, graph_ms * 1e3 / (gsteps * reps), gsteps, reps);

    cudaGraphExecDestroy(exec);
    cudaGraphDestroy(graph);
    fasgd_destroy(h);
    for (int r = 0; r < R; ++r) cudaFree(pool[r]);
    cudaStreamDestroy(stream);
    return 0;
}
