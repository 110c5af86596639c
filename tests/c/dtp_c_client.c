/*
 * A plain C client of libdtp: reads X [T,d], C [H,T,d], W_gate, W_up [N,d] (fp32, raw, in that
 * order) from argv[1], runs the first-order affinity pass and the one-layer layout search
 * through the C ABI only, and writes A [H,N] (fp32), h [H], nu [N] (int32) and score_q (int64)
 * to argv[2].  Sizes come from argv[3..7]: T d H N D.
 */
#include <stdio.h>
#include <stdlib.h>

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
    return 0;
}
