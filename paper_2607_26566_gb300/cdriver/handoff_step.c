/*
 * handoff_step.c -- the text-to-image handoff workload driven from C through
 * the store's C ABI (include/t2istore.h), with no Python between calls.
 *
 * Each of R requests in flight puts its four producer tensors (bf16 text
 * embeddings [B,512,4096], bf16 pooled embeddings [B,768], fp32 latents
 * [B,16,128,128], fp16 image [B,3,1024,1024]) with one t2i_put_batch, and
 * gets them back into consumer buffers with one t2i_get_batch, the latents
 * cast fp32 -> bf16 (§5.2: a producer writes its output into the store, a
 * consumer pulls it into its own memory). Request r runs on stream r % S;
 * the streams are joined at the two phase boundaries of a step, and a step
 * ends with one t2i_free of every object. This is the step bench.py times
 * through the Python binding: the difference between the two is the
 * binding's cost, and this program's host time per call is the library's
 * own (pointer checks, directory, page dependencies, launch).
 *
 * Usage: handoff_step B [requests streams steps warmup page_bytes pool_gib check_pointers device]
 * Prints one JSON line: GB/s of the step (algorithmic bytes: 2 x payload for
 * a put, 2 x payload for a copy and 1.5 x payload for the cast in a get) and
 * host microseconds per put and per get call. Inputs are constant bytes per
 * object; after the timed steps every copied output is compared with its
 * input byte pattern (the cast is checked bit by bit by the test suite).
 */
#define _POSIX_C_SOURCE 199309L
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <time.h>

#include "t2istore.h"

#define NOBJ 4
#define CHECK_CUDA(x)                                                                     \
    do {                                                                                  \
        cudaError_t e_ = (x);                                                             \
        if (e_ != cudaSuccess) {                                                          \
            fprintf(stderr, "%s:%d %s: %s\n", __FILE__, __LINE__, #x, cudaGetErrorString(e_)); \
            exit(2);                                                                      \
        }                                                                                 \
    } while (0)
#define CHECK_T2I(st, h, what)                                                         \
    do {                                                                               \
        if ((st) != T2I_OK) {                                                          \
            fprintf(stderr, "%s failed (%d): %s\n", what, (int)(st), t2i_last_error(h)); \
            exit(3);                                                                   \
        }                                                                              \
    } while (0)

static double now_us(void) {
    struct timespec ts;
    clock_gettime(CLOCK_MONOTONIC, &ts);
    return ts.tv_sec * 1e6 + ts.tv_nsec * 1e-3;
}

int main(int argc, char** argv) {
    if (argc < 2) {
        fprintf(stderr, "usage: %s B [requests streams steps warmup page_bytes pool_gib check_pointers device]\n",
                argv[0]);
        return 1;
    }
    const uint64_t B = strtoull(argv[1], NULL, 10);
    const int R = argc > 2 ? atoi(argv[2]) : 64;
    const int S = argc > 3 ? atoi(argv[3]) : 4;
    const int steps = argc > 4 ? atoi(argv[4]) : 50;
    const int warmup = argc > 5 ? atoi(argv[5]) : 3;
    const uint64_t page = argc > 6 ? strtoull(argv[6], NULL, 10) : (2ull << 20);
    const uint64_t pool_bytes = (argc > 7 ? strtoull(argv[7], NULL, 10) : 8ull) << 30;
    const uint32_t check_pointers = argc > 8 ? (uint32_t)atoi(argv[8]) : 1u;
    const int device = argc > 9 ? atoi(argv[9]) : 0;
    if (B < 1 || R < 1 || S < 1 || S > 64 || steps < 1 || warmup < 0 || device < 0) {
        fprintf(stderr, "bad arguments\n");
        return 1;
    }
    const uint64_t nbytes[NOBJ] = {B * 512 * 4096 * 2, B * 768 * 2, B * 16 * 128 * 128 * 4, B * 3 * 1024 * 1024 * 2};
    const int cast_obj = 2;  /* the latents */
    uint64_t payload = 0;
    for (int j = 0; j < NOBJ; ++j) payload += nbytes[j];
    const double put_bytes = 2.0 * payload * R;
    const double get_bytes = (2.0 * (payload - nbytes[cast_obj]) + 1.5 * nbytes[cast_obj]) * R;

    CHECK_CUDA(cudaSetDevice(device));
    void* pool = NULL;
    CHECK_CUDA(cudaMalloc(&pool, pool_bytes));
    t2i_store_config cfg;
    memset(&cfg, 0, sizeof cfg);
    cfg.pool_bytes = pool_bytes;
    cfg.page_bytes = page;
    cfg.check_pointers = check_pointers;
    t2i_store* h = NULL;
    t2i_status st = t2i_store_create(pool, &cfg, device, &h);
    if (st != T2I_OK) {
        fprintf(stderr, "t2i_store_create failed (%d)\n", (int)st);
        return 3;
    }

    /* producer and consumer buffers: one allocation per tensor */
    t2i_put_desc* pd = calloc((size_t)R * NOBJ, sizeof *pd);
    t2i_get_desc* gd = calloc((size_t)R * NOBJ, sizeof *gd);
    t2i_id* ids = calloc((size_t)R * NOBJ, sizeof *ids);
    void** outs = calloc((size_t)R * NOBJ, sizeof *outs);
    for (int r = 0; r < R; ++r)
        for (int j = 0; j < NOBJ; ++j) {
            const int k = r * NOBJ + j;
            void* src = NULL;
            CHECK_CUDA(cudaMalloc(&src, nbytes[j]));
            CHECK_CUDA(cudaMemset(src, (r * NOBJ + j) & 0xFF, nbytes[j]));
            const uint64_t ob = j == cast_obj ? nbytes[j] / 2 : nbytes[j];
            CHECK_CUDA(cudaMalloc(&outs[k], ob));
            pd[k].src = src;
            pd[k].nbytes = nbytes[j];
            pd[k].dtype_tag = (uint32_t)j;
            gd[k].dst = outs[k];
            gd[k].dst_bytes = ob;
            gd[k].cast = j == cast_obj;
        }
    CHECK_CUDA(cudaDeviceSynchronize());

    cudaStream_t s[64];
    cudaEvent_t done[64], hub, t0, t1;
    for (int i = 0; i < S; ++i) {
        CHECK_CUDA(cudaStreamCreateWithFlags(&s[i], cudaStreamNonBlocking));
        CHECK_CUDA(cudaEventCreateWithFlags(&done[i], cudaEventDisableTiming));
    }
    CHECK_CUDA(cudaEventCreateWithFlags(&hub, cudaEventDisableTiming));
    CHECK_CUDA(cudaEventCreate(&t0));
    CHECK_CUDA(cudaEventCreate(&t1));

    double host_put_us = 0, host_get_us = 0;
    for (int it = 0; it < warmup + steps; ++it) {
        const int timed = it >= warmup;
        if (it == warmup) {
            CHECK_CUDA(cudaDeviceSynchronize());
            CHECK_CUDA(cudaEventRecord(t0, s[0]));
            for (int i = 1; i < S; ++i) CHECK_CUDA(cudaStreamWaitEvent(s[i], t0, 0));
        }
        double a = now_us();
        for (int r = 0; r < R; ++r) {
            st = t2i_put_batch(h, pd + r * NOBJ, NOBJ, ids + r * NOBJ, s[r % S]);
            CHECK_T2I(st, h, "t2i_put_batch");
        }
        double b = now_us();
        /* join: every stream waits for all of them (through s[0]) */
        for (int i = 1; i < S; ++i) {
            CHECK_CUDA(cudaEventRecord(done[i], s[i]));
            CHECK_CUDA(cudaStreamWaitEvent(s[0], done[i], 0));
        }
        CHECK_CUDA(cudaEventRecord(hub, s[0]));
        for (int i = 1; i < S; ++i) CHECK_CUDA(cudaStreamWaitEvent(s[i], hub, 0));
        double c = now_us();
        for (int r = 0; r < R; ++r) {
            for (int j = 0; j < NOBJ; ++j) gd[r * NOBJ + j].id = ids[r * NOBJ + j];
            st = t2i_get_batch(h, gd + r * NOBJ, NOBJ, NULL, s[r % S]);
            CHECK_T2I(st, h, "t2i_get_batch");
        }
        double d = now_us();
        for (int i = 1; i < S; ++i) {
            CHECK_CUDA(cudaEventRecord(done[i], s[i]));
            CHECK_CUDA(cudaStreamWaitEvent(s[0], done[i], 0));
        }
        CHECK_CUDA(cudaEventRecord(hub, s[0]));
        for (int i = 1; i < S; ++i) CHECK_CUDA(cudaStreamWaitEvent(s[i], hub, 0));
        st = t2i_free(h, ids, (uint32_t)(R * NOBJ));
        CHECK_T2I(st, h, "t2i_free");
        if (timed) {
            host_put_us += b - a;
            host_get_us += d - c;
        }
    }
    CHECK_CUDA(cudaEventRecord(t1, s[0]));
    CHECK_CUDA(cudaEventSynchronize(t1));
    float ms = 0;
    CHECK_CUDA(cudaEventElapsedTime(&ms, t0, t1));
    CHECK_CUDA(cudaDeviceSynchronize());

    /* every copied output holds its input's byte pattern */
    int bad = 0;
    unsigned char* host = malloc(nbytes[NOBJ - 1] > nbytes[0] ? nbytes[NOBJ - 1] : nbytes[0]);
    for (int r = 0; r < R && !bad; ++r)
        for (int j = 0; j < NOBJ && !bad; ++j) {
            if (j == cast_obj) continue;
            const int k = r * NOBJ + j;
            CHECK_CUDA(cudaMemcpy(host, outs[k], nbytes[j], cudaMemcpyDeviceToHost));
            for (uint64_t i = 0; i < nbytes[j]; ++i)
                if (host[i] != (unsigned char)((r * NOBJ + j) & 0xFF)) {
                    bad = 1;
                    break;
                }
        }
    free(host);
    const double calls = (double)R * steps;
    printf("{\"B\": %llu, \"requests\": %d, \"streams\": %d, \"steps\": %d, \"page_bytes\": %llu, "
           "\"gbs\": %.1f, \"ms_per_step\": %.4f, \"host_us_per_put\": %.3f, \"host_us_per_get\": %.3f, "
           "\"check_pointers\": %u, \"outputs_ok\": %s}\n",
           (unsigned long long)B, R, S, steps, (unsigned long long)page, (put_bytes + get_bytes) * steps / (ms * 1e-3) / 1e9,
           ms / steps, host_put_us / calls, host_get_us / calls, check_pointers, bad ? "false" : "true");
    t2i_store_destroy(h);
    return bad ? 4 : 0;
}
