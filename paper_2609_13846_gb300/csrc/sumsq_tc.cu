// sumsq_tc.cu -- sums over the rows of a bf16 GEMM of its squared outputs, on
// the tcgen05 tensor cores:
//
//     out[grp, col] (+)= sum over rows r of group grp of (sum_i Arow[r, i] Bcol[col, i])^2
//
// Two uses from Sec. 3 "Affinity scores":
//   * kDown: the down-edge weight factor ||b_gk||^2 with b_gk = W^qkv_g (gamma' .
//     w^d_k): rows = the next layer's q/k/v rows of KV group g, columns = the
//     neurons (B = gamma' . W_down^T, made K-major by prep_down_weight_kernel).
//   * kAdd: the ADD score E_t[(p_h . w^g_k)^2 + (p_h . w^u_k)^2] (before the
//     mean): rows = the tokens of C_h, B = a neuron tile's W_gate rows stacked on
//     its W_up rows, and the two columns of a neuron are added.
//
// Structure as in affinity_tc.cu: persistent grid, one CTA per SM, warp 0 TMA
// producer, warp 1 MMA issuer (one 128 x 256 x 16 tcgen05.mma per K step),
// eight epilogue warps; TMEM double-buffered across units.  The epilogue sums
// the squares over its warp's 32 rows with a shuffle butterfly and over the
// four lane quadrants in shared memory in a fixed order; each unit writes its
// own partial slot and a reduce kernel adds the row chunks in order, so the
// result is deterministic.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace sq {

constexpr int BR = 128;       // rows per chunk (MMA M, TMEM lanes)
constexpr int BCOL = 256;     // MMA N
constexpr int BK = 64;
constexpr int UK = 16;
constexpr int STAGES = 4;
constexpr int kThreads = 384;
constexpr int kEpiWarps = 8;
constexpr int kEpiWarp0 = 4;
constexpr uint32_t kTileA = BR * BK * 2;          // 16 KB
constexpr uint32_t kTileB = BCOL * BK * 2;        // 32 KB
constexpr uint32_t kStageBytes = kTileA + kTileB;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBufCols = 256;
constexpr size_t kRedBytes = 2 * 4 * BCOL * sizeof(float);   // [slot][quadrant][column]
constexpr size_t kSmemBytes = 1024 + STAGES * kStageBytes + kRedBytes + 256;
constexpr uint32_t kIdesc = idesc_bf16_f32(BR, BCOL);

enum Mode { kDown = 0, kAdd = 1 };

struct Params {
    int groups;       // row groups (KV groups)
    int row_chunks;   // chunks of 128 rows per group
    int col_tiles;    // column tiles
    int KB;           // k blocks of 64
    int64_t units;    // groups * row_chunks * col_tiles
    int out_cols;     // outputs per unit: 256 (kDown) or 128 (kAdd)
    float* partial;   // [units][out_cols]
    int* status;
};

__device__ __forceinline__ float butterfly32(float (&v)[32], int lane) {
#pragma unroll
    for (int r = 0; r < 5; ++r) {
        const int o = 16 >> r;
        const int m = 16 >> r;
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < m; ++i) {
            const float send = upper ? v[i] : v[i + m];
            const float keep = upper ? v[i + m] : v[i];
            v[i] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, o);
        }
    }
    return v[0];
}

// unit u -> (group, row chunk, column tile), column tile fastest so a row chunk
// stays in L2 while it meets every column tile
__device__ __forceinline__ void decode(const Params& p, int64_t u, int& g, int& rc, int& j) {
    j = static_cast<int>(u % p.col_tiles);
    const int64_t q = u / p.col_tiles;
    rc = static_cast<int>(q % p.row_chunks);
    g = static_cast<int>(q / p.row_chunks);
}

template <int MODE>
__global__ void __launch_bounds__(kThreads, 1)
sumsq_tc_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b0,
                const __grid_constant__ CUtensorMap tm_b1, const Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    float* red = reinterpret_cast<float*>(smem + STAGES * kStageBytes);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * kStageBytes + kRedBytes);
    uint64_t* full_bar = bars;
    uint64_t* empty_bar = bars + STAGES;
    uint64_t* acc_full = bars + 2 * STAGES;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* red_full = acc_full + 4;
    uint64_t* drain_bar = acc_full + 6;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 7);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), kEpiWarps);
            mbar_init(smem_u32(&red_full[b]), kEpiWarps);
        }
        mbar_init(smem_u32(drain_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tm_a);
        tma_prefetch_desc(&tm_b0);
        tma_prefetch_desc(&tm_b1);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // -------------------------------------------------------------------- producer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t issued_parity[STAGES];
        bool issued[STAGES];
        for (int s = 0; s < STAGES; ++s) issued[s] = false, issued_parity[s] = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x) {
            int g, rc, j;
            decode(p, u, g, rc, j);
            for (int kb = 0; kb < p.KB; ++kb) {
                if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
                const uint32_t fb = smem_u32(&full_bar[stage]);
                uint8_t* st = tiles + stage * kStageBytes;
                mbar_arrive_expect_tx(fb, kStageBytes);
                tma_load_3d(smem_u32(st), &tm_a, fb, kb * BK, rc * BR, g);
                if (MODE == kDown) {
                    tma_load_2d(smem_u32(st + kTileA), &tm_b0, fb, kb * BK, j * BCOL);
                } else {
                    tma_load_2d(smem_u32(st + kTileA), &tm_b0, fb, kb * BK, j * (BCOL / 2));
                    tma_load_2d(smem_u32(st + kTileA + kTileB / 2), &tm_b1, fb, kb * BK, j * (BCOL / 2));
                }
                issued[stage] = true;
                issued_parity[stage] = phase;
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
        }
        if (!ok) {
            for (int s = 0; s < STAGES; ++s)
                if (issued[s]) {
                    const uint64_t t0 = globaltimer_ns();
                    while (!mbar_try_wait(smem_u32(&full_bar[s]), issued_parity[s]) &&
                           globaltimer_ns() - t0 < kWaitLimitNs) {
                    }
                }
        }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0, unit_count = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x, ++unit_count) {
            const uint32_t buf = unit_count & 1u;
            const uint32_t use = (unit_count >> 1) & 1u;
            if (!mbar_wait(smem_u32(&acc_empty[buf]), use ^ 1u, abort_flag)) { ok = false; break; }
            tc_fence_after();
            const uint32_t d_acc = tmem + buf * kBufCols;
            for (int kb = 0; kb < p.KB; ++kb) {
                if (!mbar_wait(smem_u32(&full_bar[stage]), phase, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t st = smem_u32(tiles + stage * kStageBytes);
                const uint64_t da = smem_desc_k128(st);
                const uint64_t db = smem_desc_k128(st + kTileA);
#pragma unroll
                for (int kk = 0; kk < BK / UK; ++kk) {
                    const uint64_t off = static_cast<uint64_t>((kk * UK * 2) >> 4);
                    umma_bf16(d_acc, da + off, db + off, kIdesc, (kb > 0 || kk > 0) ? 1u : 0u);
                }
                umma_commit(smem_u32(&empty_bar[stage]));
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            umma_commit(smem_u32(&acc_full[buf]));
        }
        umma_commit(smem_u32(drain_bar));
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(smem_u32(drain_bar), 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
    } else if (warp >= kEpiWarp0) {
        // -------------------------------------------------------------------- epilogue
        const int quad = warp & 3;
        const int half = (warp - kEpiWarp0) >> 2;
        const bool summer = (quad == 0);
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
        // kDown: this warp owns output columns [128*half, 128*half + 128) (4 blocks of 32)
        // kAdd : output neurons [64*half, 64*half + 64) (2 blocks), gate col n, up col 128 + n
        constexpr int kBlocks = MODE == kDown ? 4 : 2;
        constexpr int kPerHalf = 32 * kBlocks;
        uint32_t unit_count = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x, ++unit_count) {
            const uint32_t buf = unit_count & 1u;
            const uint32_t use = (unit_count >> 1) & 1u;
            if (!mbar_wait(smem_u32(&acc_full[buf]), use, abort_flag)) { ok = false; break; }
            tc_fence_after();
            const uint32_t acc = lane_base + buf * kBufCols;
            float colsum[kBlocks];
#pragma unroll
            for (int blk = 0; blk < kBlocks; ++blk) {
                float v[32];
                if (MODE == kDown) {
                    const uint32_t c0 = static_cast<uint32_t>(128 * half + 32 * blk);
                    tmem_ld16(acc + c0, &v[0]);
                    tmem_ld16(acc + c0 + 16u, &v[16]);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) v[e] = v[e] * v[e];
                } else {
                    float w[32];
                    const uint32_t c0 = static_cast<uint32_t>(64 * half + 32 * blk);
                    tmem_ld16(acc + c0, &v[0]);
                    tmem_ld16(acc + c0 + 16u, &v[16]);
                    tmem_ld16(acc + 128u + c0, &w[0]);
                    tmem_ld16(acc + 128u + c0 + 16u, &w[16]);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) v[e] = fmaf(v[e], v[e], w[e] * w[e]);
                }
                colsum[blk] = butterfly32(v, lane);
            }
            const uint32_t slot = unit_count & 1u;
            const uint32_t rphase = (unit_count >> 1) & 1u;
            float* rs = red + slot * 4 * BCOL;
            if (!summer) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_empty[buf]));
            }
#pragma unroll
            for (int blk = 0; blk < kBlocks; ++blk) rs[quad * BCOL + kPerHalf * half + 32 * blk + lane] = colsum[blk];
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&red_full[slot]));
            if (summer) {
                if (!mbar_wait(smem_u32(&red_full[slot]), rphase, abort_flag)) { ok = false; break; }
                float* o = p.partial + u * p.out_cols + kPerHalf * half;
#pragma unroll
                for (int blk = 0; blk < kBlocks; ++blk) {
                    const int n = kPerHalf * half + 32 * blk + lane;
                    o[32 * blk + lane] = ((rs[n] + rs[BCOL + n]) + rs[2 * BCOL + n]) + rs[3 * BCOL + n];
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&acc_empty[buf]));
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, static_cast<int>(DTP_ERR_NOT_CONVERGED));
}

// out[g, col] (+)= sum over row chunks (in order) of the unit partials; col < n_cols.
// out row o sums groups o*qpg .. o*qpg + qpg - 1 (group by group, then row chunks).
__global__ void sumsq_reduce_kernel(const float* __restrict__ partial, float* __restrict__ out, int groups,
                                    int row_chunks, int col_tiles, int out_cols, int n_cols, int accumulate, int qpg) {
    const int64_t total = static_cast<int64_t>(groups / qpg) * n_cols;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int o = static_cast<int>(idx / n_cols);
        const int col = static_cast<int>(idx % n_cols);
        const int j = col / out_cols, r = col % out_cols;
        float s = 0.0f;
        for (int g = o * qpg; g < (o + 1) * qpg; ++g)
            for (int rc = 0; rc < row_chunks; ++rc)
                s += partial[((static_cast<int64_t>(g) * row_chunks + rc) * col_tiles + j) * out_cols + r];
        out[idx] = accumulate ? out[idx] + s : s;
    }
}

// WdT[k, i] = bf16(gamma[i] * W_down[i, k]): gamma' . w^d_k as K-major rows.
template <typename T>
__global__ void prep_down_weight_kernel(const T* __restrict__ Wd, const T* __restrict__ gamma, int d, int N,
                                        __nv_bfloat16* __restrict__ WdT) {
    __shared__ float tile[32][33];
    const int i0 = blockIdx.y * 32, k0 = blockIdx.x * 32;
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int i = i0 + r, k = k0 + threadIdx.x;
        tile[r][threadIdx.x] = (i < d && k < N) ? static_cast<float>(gamma[i]) * static_cast<float>(Wd[static_cast<int64_t>(i) * N + k]) : 0.0f;
    }
    __syncthreads();
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int k = k0 + r, i = i0 + threadIdx.x;
        if (k < N && i < d) WdT[static_cast<int64_t>(k) * d + i] = __float2bfloat16_rn(tile[threadIdx.x][r]);
    }
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

static bool map_bf16(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides,
                     cuuint32_t box_rows) {
    auto enc = encode_fn();
    if (!enc) return false;
    cuuint32_t box[3] = {static_cast<cuuint32_t>(BK), box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int MODE>
static int run(const CUtensorMap& ma, const CUtensorMap& mb0, const CUtensorMap& mb1, Params p, float* out,
               int n_cols, int accumulate, cudaStream_t stream, int qpg = 1) {
    int dev = 0, sms = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaFuncSetAttribute(sumsq_tc_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBytes)));
    const int grid = static_cast<int>(p.units < sms ? p.units : sms);
    sumsq_tc_kernel<MODE><<<grid, kThreads, kSmemBytes, stream>>>(ma, mb0, mb1, p);
    DTP_CUDA_TRY(cudaGetLastError());
    const int64_t total = static_cast<int64_t>(p.groups / qpg) * n_cols;
    const int blocks = static_cast<int>((total + 255) / 256 < 4 * sms ? (total + 255) / 256 : 4 * sms);
    sumsq_reduce_kernel<<<blocks, 256, 0, stream>>>(p.partial, out, p.groups, p.row_chunks, p.col_tiles, p.out_cols,
                                                    n_cols, accumulate, qpg);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

// ---------------------------------------------------------------- down edge --

size_t down_workspace_bytes(int G, int R, int d, int N) {
    const int64_t units = static_cast<int64_t>(G) * ((R + BR - 1) / BR) * ((N + BCOL - 1) / BCOL);
    return kWorkspaceHeader + align_up(static_cast<size_t>(N) * d * 2, 256) +
           static_cast<size_t>(units) * BCOL * sizeof(float);
}

int launch_down(const void* Wqkv, const void* gamma, const void* Wd, int G, int R, int d, int N, int dtype, float* bn,
                void* workspace, cudaStream_t stream) {
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
    __nv_bfloat16* WdT = reinterpret_cast<__nv_bfloat16*>(ws + kWorkspaceHeader);
    float* partial = reinterpret_cast<float*>(ws + kWorkspaceHeader + align_up(static_cast<size_t>(N) * d * 2, 256));
    dim3 pb(32, 8), pg((N + 31) / 32, (d + 31) / 32);
    if (dtype == DTP_BF16)
        prep_down_weight_kernel<__nv_bfloat16><<<pg, pb, 0, stream>>>(static_cast<const __nv_bfloat16*>(Wd),
                                                                      static_cast<const __nv_bfloat16*>(gamma), d, N, WdT);
    else
        prep_down_weight_kernel<float><<<pg, pb, 0, stream>>>(static_cast<const float*>(Wd),
                                                              static_cast<const float*>(gamma), d, N, WdT);
    DTP_CUDA_TRY(cudaGetLastError());
    CUtensorMap ma, mb;
    const cuuint64_t rs = static_cast<cuuint64_t>(d) * 2;
    cuuint64_t da[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(R), static_cast<cuuint64_t>(G)};
    cuuint64_t sa[2] = {rs, rs * static_cast<cuuint64_t>(R)};
    cuuint64_t db[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N)};
    cuuint64_t sb[1] = {rs};
    if (!map_bf16(&ma, Wqkv, 3, da, sa, BR) || !map_bf16(&mb, WdT, 2, db, sb, BCOL)) return DTP_ERR_CUDA;
    Params p;
    p.groups = G;
    p.row_chunks = (R + BR - 1) / BR;
    p.col_tiles = (N + BCOL - 1) / BCOL;
    p.KB = (d + BK - 1) / BK;
    p.units = static_cast<int64_t>(p.groups) * p.row_chunks * p.col_tiles;
    p.out_cols = BCOL;
    p.partial = partial;
    p.status = reinterpret_cast<int*>(ws);
    return run<kDown>(ma, mb, mb, p, bn, N, 0, stream);
}

// ---------------------------------------------------------------- ADD score --

size_t add_workspace_bytes(int64_t T, int G, int N) {
    const int64_t units = static_cast<int64_t>(G) * ((T + BR - 1) / BR) * ((N + 127) / 128);
    return kWorkspaceHeader + static_cast<size_t>(units) * 128 * sizeof(float);
}

// G heads of C; A_add receives G / qpg rows (qpg consecutive heads summed per row).
int launch_add_grouped(const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A_add,
                       void* workspace, cudaStream_t stream, int qpg) {
    if (qpg < 1 || G % qpg) return DTP_ERR_ARG;
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
    CUtensorMap mc, mg, mu;
    const cuuint64_t rs = static_cast<cuuint64_t>(d) * 2;
    cuuint64_t dc[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(G)};
    cuuint64_t sc[2] = {rs, rs * static_cast<cuuint64_t>(T)};
    cuuint64_t dw[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N)};
    cuuint64_t sw[1] = {rs};
    if (!map_bf16(&mc, C, 3, dc, sc, BR) || !map_bf16(&mg, Wg, 2, dw, sw, BCOL / 2) ||
        !map_bf16(&mu, Wu, 2, dw, sw, BCOL / 2))
        return DTP_ERR_CUDA;
    Params p;
    p.groups = G;
    p.row_chunks = static_cast<int>((T + BR - 1) / BR);
    p.col_tiles = (N + 127) / 128;
    p.KB = (d + BK - 1) / BK;
    p.units = static_cast<int64_t>(p.groups) * p.row_chunks * p.col_tiles;
    p.out_cols = 128;
    p.partial = reinterpret_cast<float*>(ws + kWorkspaceHeader);
    p.status = reinterpret_cast<int*>(ws);
    return run<kAdd>(mc, mg, mu, p, A_add, N, 1, stream, qpg);
}

int launch_add(const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A_add,
               void* workspace, cudaStream_t stream) {
    return launch_add_grouped(C, Wg, Wu, T, d, G, N, A_add, workspace, stream, 1);
}

}  // namespace sq
}  // namespace dtp
