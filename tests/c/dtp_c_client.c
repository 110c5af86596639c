/*
 * A plain C client of libdtp: reads X [T,d], C [H,T,d], W_gate, W_up [N,d] (fp32, raw, in that
 * order) from argv[1], runs the first-order affinity pass and the one-layer layout search
 * through the C ABI only, and writes A [H,N] (fp32), h [H], nu [N] (int32) and score_q (int64)
 * to argv[2].  Sizes come from argv[3..7]: T d H N D.  It then rounds the inputs to bf16 and runs
 * the bf16 pass twice, with a workspace and through the allocation-free entry point, and prints
 * whether the two results are equal bit for bit and the allocation-free call's device status.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime.h>

#include "dtp.h"

#define CHECK(call)                                                             \
    do {                                                                        \
        int st_ = (int)(call);                                                  \
        if (st_ != 0) {                                                         \
            fprintf(stderr, "%s failed: %d (%s)\n", #call, st_, dtp_status_string(st_)); \
            return 1;                                                           \
        }                                                                       \
    } while (0)

/* fp32 -> bf16, round to nearest even (finite inputs) */
static uint16_t to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static int read_all(const char* path, float* dst, size_t n) {
    FILE* f = fopen(path, "rb");
    if (!f) return 1;
    size_t got = fread(dst, sizeof(float), n, f);
    fclose(f);
    return got == n ? 0 : 1;
}

int main(int argc, char** argv) {
    if (argc != 8) {
        fprintf(stderr, "usage: %s in.bin out.bin T d H N D\n", argv[0]);
        return 2;
    }
    const long long T = atoll(argv[3]);
    const int d = atoi(argv[4]), H = atoi(argv[5]), N = atoi(argv[6]), D = atoi(argv[7]);
    const size_t nx = (size_t)T * d, nc = (size_t)H * T * d, nw = (size_t)N * d;
    float* host = (float*)malloc(sizeof(float) * (nx + nc + 2 * nw));
    if (!host || read_all(argv[1], host, nx + nc + 2 * nw)) return 3;

    float *x, *c, *wg, *wu, *a;
    int32_t *h, *nu, *iters;
    int64_t* score_q;
    double* score;
    void *ws_aff, *ws_search;
    size_t b_aff = 0, b_search = 0;
    CHECK(dtp_affinity_workspace_size(T, d, H, N, DTP_F32, &b_aff));
    CHECK(dtp_search_workspace_size(1, H, N, D, &b_search));
    CHECK(cudaMalloc((void**)&x, sizeof(float) * nx));
    CHECK(cudaMalloc((void**)&c, sizeof(float) * nc));
    CHECK(cudaMalloc((void**)&wg, sizeof(float) * nw));
    CHECK(cudaMalloc((void**)&wu, sizeof(float) * nw));
    CHECK(cudaMalloc((void**)&a, sizeof(float) * (size_t)H * N));
    CHECK(cudaMalloc((void**)&h, sizeof(int32_t) * H));
    CHECK(cudaMalloc((void**)&nu, sizeof(int32_t) * N));
    CHECK(cudaMalloc((void**)&iters, sizeof(int32_t)));
    CHECK(cudaMalloc((void**)&score_q, sizeof(int64_t)));
    CHECK(cudaMalloc((void**)&score, sizeof(double)));
    CHECK(cudaMalloc(&ws_aff, b_aff));
    CHECK(cudaMalloc(&ws_search, b_search));
    CHECK(cudaMemcpy(x, host, sizeof(float) * nx, cudaMemcpyHostToDevice));
    CHECK(cudaMemcpy(c, host + nx, sizeof(float) * nc, cudaMemcpyHostToDevice));
    CHECK(cudaMemcpy(wg, host + nx + nc, sizeof(float) * nw, cudaMemcpyHostToDevice));
    CHECK(cudaMemcpy(wu, host + nx + nc + nw, sizeof(float) * nw, cudaMemcpyHostToDevice));
    CHECK(cudaMemset(a, 0, sizeof(float) * (size_t)H * N));

    CHECK(dtp_affinity_accumulate(x, c, wg, wu, T, d, H, N, DTP_F32, a, ws_aff, b_aff, NULL));
    CHECK(dtp_search_layout(a, H, N, D, 10, h, nu, score_q, score, iters, ws_search, b_search, NULL));
    CHECK(cudaDeviceSynchronize());
    CHECK(dtp_workspace_status(ws_aff, b_aff, NULL));
    CHECK(dtp_workspace_status(ws_search, b_search, NULL));

    float* A = (float*)malloc(sizeof(float) * (size_t)H * N);
    int32_t* hh = (int32_t*)malloc(sizeof(int32_t) * H);
    int32_t* nn = (int32_t*)malloc(sizeof(int32_t) * N);
    int64_t sq = 0;
    CHECK(cudaMemcpy(A, a, sizeof(float) * (size_t)H * N, cudaMemcpyDeviceToHost));
    CHECK(cudaMemcpy(hh, h, sizeof(int32_t) * H, cudaMemcpyDeviceToHost));
    CHECK(cudaMemcpy(nn, nu, sizeof(int32_t) * N, cudaMemcpyDeviceToHost));
    CHECK(cudaMemcpy(&sq, score_q, sizeof(int64_t), cudaMemcpyDeviceToHost));
    FILE* f = fopen(argv[2], "wb");
    if (!f) return 4;
    fwrite(A, sizeof(float), (size_t)H * N, f);
    fwrite(hh, sizeof(int32_t), H, f);
    fwrite(nn, sizeof(int32_t), N, f);
    fwrite(&sq, sizeof(int64_t), 1, f);
    fclose(f);
    printf("ok %lld\n", (long long)sq);

    /* bf16: the workspace entry point and the allocation-free one on the same inputs */
    const size_t ntot = nx + nc + 2 * nw;
    uint16_t* hb = (uint16_t*)malloc(sizeof(uint16_t) * ntot);
    if (!hb) return 3;
    for (size_t i = 0; i < ntot; ++i) hb[i] = to_bf16(host[i]);
    uint16_t* xb;
    float *a_ws, *a_na;
    void* ws_bf = NULL;
    size_t b_bf = 0;
    CHECK(dtp_affinity_workspace_size(T, d, H, N, DTP_BF16, &b_bf));
    CHECK(cudaMalloc((void**)&xb, sizeof(uint16_t) * ntot));
    CHECK(cudaMalloc((void**)&a_ws, sizeof(float) * (size_t)H * N));
    CHECK(cudaMalloc((void**)&a_na, sizeof(float) * (size_t)H * N));
    CHECK(cudaMalloc(&ws_bf, b_bf));
    CHECK(cudaMemcpy(xb, hb, sizeof(uint16_t) * ntot, cudaMemcpyHostToDevice));
    CHECK(cudaMemset(a_ws, 0, sizeof(float) * (size_t)H * N));
    CHECK(cudaMemset(a_na, 0, sizeof(float) * (size_t)H * N));
    CHECK(dtp_affinity_accumulate(xb, xb + nx, xb + nx + nc, xb + nx + nc + nw, T, d, H, N, DTP_BF16, a_ws, ws_bf,
                                  b_bf, NULL));
    CHECK(dtp_affinity_accumulate_noalloc(xb, xb + nx, xb + nx + nc, xb + nx + nc + nw, T, d, H, N, a_na, NULL));
    const int na_status = dtp_affinity_noalloc_status(NULL);
    CHECK(cudaDeviceSynchronize());
    CHECK(dtp_workspace_status(ws_bf, b_bf, NULL));
    float* A1 = (float*)malloc(sizeof(float) * (size_t)H * N);
    float* A2 = (float*)malloc(sizeof(float) * (size_t)H * N);
    if (!A1 || !A2) return 3;
    CHECK(cudaMemcpy(A1, a_ws, sizeof(float) * (size_t)H * N, cudaMemcpyDeviceToHost));
    CHECK(cudaMemcpy(A2, a_na, sizeof(float) * (size_t)H * N, cudaMemcpyDeviceToHost));
    printf("noalloc_equal %d status %d\n", memcmp(A1, A2, sizeof(float) * (size_t)H * N) == 0, na_status);
    return 0;
}
