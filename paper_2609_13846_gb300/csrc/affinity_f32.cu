// affinity_f32.cu -- fp32 mode of the first-order affinity (Sec. 3 "Affinity
// scores") on the CUDA cores, plus the finalize and ||w^d||^2 helpers.
//
// The fp32 mode exists for tight checks (fp32 operands, fp32 FMA); TF32
// tensor cores would not meet a 1e-5 relative error.  A block computes a
// 64-token x 64-neuron tile: the X pass gives (alpha, beta) per (token, neuron)
// in registers, then each head pass gives (pg, pu) and Delta^2 is summed over
// the block's tokens.  Per-tile partials go to the workspace and are added
// into A in a fixed order, so the result is deterministic.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace f32 {

constexpr int TT = 64;   // tokens per tile
constexpr int TN = 64;   // neurons per tile
constexpr int TK = 16;   // k chunk
constexpr int kThreads = 256;

// acc_g[i][j] = sum_k act[t_i,k] Wg[n_j,k], acc_u likewise, for the thread's
// tokens t_i = t0 + ty + 16 i and neurons n_j = n0 + tx + 16 j.
__device__ __forceinline__ void tile_gemm(const float* __restrict__ act, int64_t T, int d,
                                          const float* __restrict__ Wg, const float* __restrict__ Wu, int N,
                                          int64_t t0, int n0, float (&acc_g)[4][4], float (&acc_u)[4][4],
                                          float (*xs)[TT + 1], float (*gs)[TN + 1], float (*us)[TN + 1]) {
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc_g[i][j] = 0.0f, acc_u[i][j] = 0.0f;
    for (int k0 = 0; k0 < d; k0 += TK) {
        // 64 rows x 16 k per operand: 1024 elements, 4 per thread
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int idx = threadIdx.x + e * kThreads;
            const int r = idx / TK, kk = idx % TK;
            const int k = k0 + kk;
            const int64_t t = t0 + r;
            const int n = n0 + r;
            xs[kk][r] = (t < T && k < d) ? act[t * d + k] : 0.0f;
            gs[kk][r] = (n < N && k < d) ? Wg[static_cast<int64_t>(n) * d + k] : 0.0f;
            us[kk][r] = (n < N && k < d) ? Wu[static_cast<int64_t>(n) * d + k] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < TK; ++kk) {
            float a[4], bg[4], bu[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = xs[kk][ty + 16 * i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bg[j] = gs[kk][tx + 16 * j], bu[j] = us[kk][tx + 16 * j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    acc_g[i][j] = fmaf(a[i], bg[j], acc_g[i][j]);
                    acc_u[i][j] = fmaf(a[i], bu[j], acc_u[i][j]);
                }
        }
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kThreads)
affinity_fo_f32_kernel(const float* __restrict__ X, const float* __restrict__ C, const float* __restrict__ Wg,
                       const float* __restrict__ Wu, int64_t T, int d, int G, int N, float* __restrict__ partial,
                       const float* __restrict__ rms, float* __restrict__ partial_act) {
    __shared__ float xs[TK][TT + 1];
    __shared__ float gs[TK][TN + 1];
    __shared__ float us[TK][TN + 1];
    __shared__ float red[16][TN + 1];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int n0 = blockIdx.x * TN;
    const int64_t tile = blockIdx.y;
    const int64_t t0 = tile * TT;

    float acc_g[4][4], acc_u[4][4], alpha[4][4], beta[4][4];
    tile_gemm(X, T, d, Wg, Wu, N, t0, n0, acc_g, acc_u, xs, gs, us);
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float g = acc_g[i][j], u = acc_u[i][j];
            const float s = 1.0f / (1.0f + expf(-g));
            beta[i][j] = g * s;
            alpha[i][j] = s * (1.0f + g * (1.0f - s)) * u;
        }
    if (rms) {
        // down-edge activation term: sum over this tile's tokens of (silu(g) u)^2 / r'^2
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float s = 0.0f;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t t = t0 + ty + 16 * i;
                if (t < T) {
                    const float act = beta[i][j] * acc_u[i][j];
                    const float r = rms[t];
                    s = fmaf(act * act, 1.0f / (r * r), s);
                }
            }
            red[ty][tx + 16 * j] = s;
        }
        __syncthreads();
        if (threadIdx.x < TN) {
            float s = 0.0f;
            for (int r = 0; r < 16; ++r) s += red[r][threadIdx.x];
            const int n = n0 + threadIdx.x;
            if (n < N) partial_act[tile * N + n] = s;
        }
        __syncthreads();
    }
    for (int h = 0; h < G; ++h) {
        tile_gemm(C + static_cast<int64_t>(h) * T * d, T, d, Wg, Wu, N, t0, n0, acc_g, acc_u, xs, gs, us);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float s = 0.0f;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float dlt = alpha[i][j] * acc_g[i][j] + beta[i][j] * acc_u[i][j];
                s = fmaf(dlt, dlt, s);
            }
            red[ty][tx + 16 * j] = s;
        }
        __syncthreads();
        if (threadIdx.x < TN) {
            float s = 0.0f;
            for (int r = 0; r < 16; ++r) s += red[r][threadIdx.x];
            const int n = n0 + threadIdx.x;
            if (n < N) partial[(tile * G + h) * N + n] = s;
        }
        __syncthreads();
    }
}

// A[g,k] += sum over heads h of row g (qpg consecutive heads) and token tiles, head by head.
__global__ void f32_reduce_kernel(const float* __restrict__ partial, float* __restrict__ A, int G, int N,
                                  int64_t tiles, const float* __restrict__ partial_act, float* __restrict__ act2,
                                  int qpg) {
    const int64_t heads_n = static_cast<int64_t>(G) * N;
    const int64_t total_a = static_cast<int64_t>(G / qpg) * N;
    const int64_t total = total_a + (act2 ? N : 0);
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        float s = 0.0f;
        if (idx < total_a) {
            const int64_t g = idx / N, k = idx % N;
            for (int64_t h = g * qpg; h < (g + 1) * qpg; ++h)
                for (int64_t t = 0; t < tiles; ++t) s += partial[t * heads_n + h * N + k];
            A[idx] += s;
        } else {
            const int64_t k = idx - total_a;
            for (int64_t t = 0; t < tiles; ++t) s += partial_act[t * N + k];
            act2[k] += s;
        }
    }
}

size_t workspace_bytes(int64_t T, int d, int G, int N) {
    (void)d;
    const int64_t tiles = (T + TT - 1) / TT;
    return kWorkspaceHeader + static_cast<size_t>(tiles) * (G + 1) * N * sizeof(float);
}

int launch_grouped(const float* X, const float* C, const float* Wg, const float* Wu, int64_t T, int d, int G, int N,
                   float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2, int qpg) {
    if (qpg < 1 || G % qpg) return DTP_ERR_ARG;
    const int64_t tiles = (T + TT - 1) / TT;
    if (tiles > 65535) return DTP_ERR_UNSUPPORTED;
    float* partial = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(workspace) + kWorkspaceHeader);
    float* partial_act = partial + tiles * static_cast<int64_t>(G) * N;
    const bool want_act = rms && act2;
    dim3 grid((N + TN - 1) / TN, static_cast<unsigned>(tiles));
    affinity_fo_f32_kernel<<<grid, kThreads, 0, stream>>>(X, C, Wg, Wu, T, d, G, N, partial,
                                                          want_act ? rms : nullptr, partial_act);
    DTP_CUDA_TRY(cudaGetLastError());
    const int64_t total = static_cast<int64_t>(G / qpg) * N + (want_act ? N : 0);
    const int blocks = static_cast<int>((total + 255) / 256 < 1024 ? (total + 255) / 256 : 1024);
    f32_reduce_kernel<<<blocks, 256, 0, stream>>>(partial, A, G, N, tiles, partial_act, want_act ? act2 : nullptr,
                                                  qpg);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

int launch(const float* X, const float* C, const float* Wg, const float* Wu, int64_t T, int d, int G, int N,
           float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2) {
    return launch_grouped(X, C, Wg, Wu, T, d, G, N, A, workspace, stream, rms, act2, 1);
}

// S_down[g,k] = act2[k] / T_total * bn[g,k]
__global__ void down_finalize_kernel(const float* __restrict__ act2, const float* __restrict__ bn, int G, int N,
                                     float inv_t, float* __restrict__ S) {
    const int64_t total = static_cast<int64_t>(G) * N;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x)
        S[idx] = act2[idx % N] * inv_t * bn[idx];
}

}  // namespace f32

// --------------------------------------------------------------------------
// finalize: A[h,k] *= wd_sqnorm[k] / T_total
// --------------------------------------------------------------------------
__global__ void finalize_kernel(float* __restrict__ A, int G, int N, float inv_t, const float* __restrict__ wd) {
    const int64_t total = static_cast<int64_t>(G) * N;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int k = static_cast<int>(idx % N);
        const float f = wd ? wd[k] : 1.0f;
        A[idx] = A[idx] * f * inv_t;
    }
}

// out[k] = sum_i W_down[i,k]^2 over the d rows of W_down [d, N].
template <typename T>
__global__ void down_sqnorm_kernel(const T* __restrict__ W, int d, int N, float* __restrict__ out) {
    const int k = blockIdx.x * blockDim.x + threadIdx.x;
    if (k >= N) return;
    float s = 0.0f;
    for (int i = 0; i < d; ++i) {
        const float w = static_cast<float>(W[static_cast<int64_t>(i) * N + k]);
        s = fmaf(w, w, s);
    }
    out[k] = s;
}

int launch_down_finalize(const float* act2, const float* bn, int G, int N, int64_t T_total, float* S,
                         cudaStream_t stream) {
    const int64_t total = static_cast<int64_t>(G) * N;
    const int blocks = static_cast<int>((total + 255) / 256 < 1024 ? (total + 255) / 256 : 1024);
    f32::down_finalize_kernel<<<blocks, 256, 0, stream>>>(act2, bn, G, N,
                                                         static_cast<float>(1.0 / static_cast<double>(T_total)), S);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

// Top-group share of each layer (Sec. 5 diagnostic): the mean over neurons with a non-zero column of
// max_g A[g,k] / sum_g A[g,k], in fp64.  One block per layer; the per-thread sums are combined in a
// fixed order (warp butterflies, then the warps in index order), so the result is reproducible.
__global__ void __launch_bounds__(1024) top_share_kernel(const float* __restrict__ A, int G, int N,
                                                         double* __restrict__ share) {
    __shared__ double ssum[32];
    __shared__ int scnt[32];
    const float* a = A + static_cast<int64_t>(blockIdx.x) * G * N;
    double acc = 0.0;
    int cnt = 0;
    for (int k = threadIdx.x; k < N; k += blockDim.x) {
        double tot = 0.0, mx = 0.0;
        for (int g = 0; g < G; ++g) {
            const double v = a[static_cast<int64_t>(g) * N + k];
            tot += v;
            mx = v > mx ? v : mx;
        }
        if (tot > 0.0) {
            acc += mx / tot;
            ++cnt;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
        cnt += __shfl_xor_sync(0xFFFFFFFFu, cnt, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) ssum[warp] = acc, scnt[warp] = cnt;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        int c = 0;
        for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += ssum[w], c += scnt[w];
        share[blockIdx.x] = c ? t / c : 0.0;
    }
}

int launch_top_share(const float* A, int layers, int G, int N, double* share, cudaStream_t stream) {
    top_share_kernel<<<layers, 1024, 0, stream>>>(A, G, N, share);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

int launch_finalize(float* A, int G, int N, int64_t T_total, const float* wd, cudaStream_t stream) {
    const int64_t total = static_cast<int64_t>(G) * N;
    const int blocks = static_cast<int>((total + 255) / 256 < 1024 ? (total + 255) / 256 : 1024);
    finalize_kernel<<<blocks, 256, 0, stream>>>(A, G, N, static_cast<float>(1.0 / static_cast<double>(T_total)), wd);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

int launch_down_sqnorm(const void* W, int d, int N, int dtype, float* out, cudaStream_t stream) {
    const int blocks = (N + 255) / 256;
    if (dtype == DTP_BF16)
        down_sqnorm_kernel<__nv_bfloat16><<<blocks, 256, 0, stream>>>(static_cast<const __nv_bfloat16*>(W), d, N, out);
    else
        down_sqnorm_kernel<float><<<blocks, 256, 0, stream>>>(static_cast<const float*>(W), d, N, out);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace dtp
