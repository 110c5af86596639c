// affinity_tc.cu -- first-order head->neuron affinity on the tcgen05 tensor
// cores (bf16 operands, fp32 accumulation), Sec. 3 "Affinity scores":
//
//     A[h,k] += sum_t ( silu'(g_tk) u_tk pg_thk + silu(g_tk) pu_thk )^2
//
// with g = X W_gate^T, u = X W_up^T (the operating point) and pg = C_h W_gate^T,
// pu = C_h W_up^T (head h's piece projected through the FFN input weights).
//
// Orientation.  The MMA's M dimension is the neuron (128 neurons of one tile
// in the 128 TMEM lanes) and its N dimension is the token (a chunk of 128
// tokens in TMEM columns).  Each epilogue thread therefore owns one neuron
// and sums Delta^2 over tokens inside its own registers: the token reduction
// needs no shuffles, and the T x G x N intermediate never leaves the SM.
//
// Work unit = (token chunk c, neuron tile j); a unit runs G+1 passes over d:
// pass 0 multiplies the X chunk, pass 1+h the C_h chunk, each against the
// tile's W_gate and W_up rows (two M=128, N=128 MMAs per K step sharing the
// activation operand).  Units are dealt round-robin to a persistent grid in
// token-chunk-major order, so the CTAs in flight share a handful of token
// chunks in L2 while all weights stay L2-resident.
//
// TMEM (512 columns x 128 lanes, fp32):
//     [  0,128) gate accumulator of the current head pass  (pg)
//     [128,256) up accumulator of the current head pass    (pu)
//     [256,384) g of pass 0, converted in place to alpha = silu'(g) u
//     [384,512) u of pass 0, converted in place to beta  = silu(g)
//
// Warp roles (320 threads): warp 0 issues TMA loads, warp 1 allocates TMEM
// and issues the MMAs (one thread), warps 2..9 are the epilogue (two warps
// per TMEM lane quadrant, each taking 64 of the 128 token columns).
//
// Determinism: every unit writes its per-(half, head, neuron) partial sums to
// its own workspace slot; a second kernel adds them into A in a fixed order.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace tc {

constexpr int BM = 128;       // neurons per tile (MMA M)
constexpr int BN = 128;       // tokens per chunk (MMA N)
constexpr int BK = 64;        // bf16 elements per 128-byte swizzled row
constexpr int UK = 16;        // K of one tcgen05.mma kind::f16
constexpr int STAGES = 4;
constexpr int kThreads = 320;
constexpr int kEpiWarps = 8;
constexpr uint32_t kTileA = BM * BK * 2;   // 16 KB, one weight operand
constexpr uint32_t kTileB = BN * BK * 2;   // 16 KB, activation operand
constexpr uint32_t kStageBytes = 2 * kTileA + kTileB;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColPg = 0, kColPu = 128, kColAlpha = 256, kColBeta = 384;
constexpr size_t kSmemBytes = 1024 + STAGES * kStageBytes + 256;
constexpr uint32_t kIdesc = idesc_bf16_f32(BM, BN);

struct Params {
    int G;          // KV heads
    int NT;         // neuron tiles
    int TC;         // token chunks
    int KB;         // k blocks of 64 over d
    int64_t units;  // NT * TC
    float* partial; // [units][2][G][128]
    int* status;    // workspace status word
};

__global__ void __launch_bounds__(kThreads, 1)
affinity_fo_tc_kernel(const __grid_constant__ CUtensorMap tm_wg, const __grid_constant__ CUtensorMap tm_wu,
                      const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_c,
                      const Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * kStageBytes);
    // bars[0..S) full, bars[S..2S) empty, then acc_full, acc_empty, ab_full, ab_empty
    uint64_t* full_bar = bars;
    uint64_t* empty_bar = bars + STAGES;
    uint64_t* acc_full = bars + 2 * STAGES;
    uint64_t* acc_empty = acc_full + 1;
    uint64_t* ab_full = acc_full + 2;
    uint64_t* ab_empty = acc_full + 3;
    uint64_t* drain_bar = acc_full + 4;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 5);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        mbar_init(smem_u32(acc_full), 1);
        mbar_init(smem_u32(acc_empty), kEpiWarps);
        mbar_init(smem_u32(ab_full), 1);
        mbar_init(smem_u32(ab_empty), kEpiWarps);
        mbar_init(smem_u32(drain_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tm_wg);
        tma_prefetch_desc(&tm_wu);
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_c);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const int passes = p.G + 1;
    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_parity[STAGES];
            bool issued[STAGES];
            for (int s = 0; s < STAGES; ++s) issued[s] = false, issued_parity[s] = 0;
            bool ok = true;
            for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x) {
                const int c = static_cast<int>(u / p.NT);
                const int j = static_cast<int>(u % p.NT);
                for (int pass = 0; ok && pass < passes; ++pass) {
                    for (int kb = 0; kb < p.KB; ++kb) {
                        if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
                        const uint32_t fb = smem_u32(&full_bar[stage]);
                        uint8_t* st = tiles + stage * kStageBytes;
                        mbar_arrive_expect_tx(fb, kStageBytes);
                        tma_load_2d(smem_u32(st), &tm_wg, fb, kb * BK, j * BM);
                        tma_load_2d(smem_u32(st + kTileA), &tm_wu, fb, kb * BK, j * BM);
                        if (pass == 0)
                            tma_load_2d(smem_u32(st + 2 * kTileA), &tm_x, fb, kb * BK, c * BN);
                        else
                            tma_load_3d(smem_u32(st + 2 * kTileA), &tm_c, fb, kb * BK, c * BN, pass - 1);
                        issued[stage] = true;
                        issued_parity[stage] = phase;
                        if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                    }
                }
            }
            if (!ok) {
                // Let copies already in flight land before the CTA exits.
                for (int s = 0; s < STAGES; ++s)
                    if (issued[s]) {
                        const uint64_t t0 = globaltimer_ns();
                        while (!mbar_try_wait(smem_u32(&full_bar[s]), issued_parity[s]) &&
                               globaltimer_ns() - t0 < kWaitLimitNs) {
                        }
                    }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0, acc_phase = 0, ab_phase = 0;
            bool ok = true;
            for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x) {
                for (int pass = 0; ok && pass < passes; ++pass) {
                    uint32_t d_gate, d_up;
                    if (pass == 0) {
                        if (!mbar_wait(smem_u32(ab_empty), ab_phase ^ 1u, abort_flag)) { ok = false; break; }
                        ab_phase ^= 1u;
                        d_gate = tmem + kColAlpha;
                        d_up = tmem + kColBeta;
                    } else {
                        if (!mbar_wait(smem_u32(acc_empty), acc_phase ^ 1u, abort_flag)) { ok = false; break; }
                        acc_phase ^= 1u;
                        d_gate = tmem + kColPg;
                        d_up = tmem + kColPu;
                    }
                    tc_fence_after();
                    for (int kb = 0; kb < p.KB; ++kb) {
                        if (!mbar_wait(smem_u32(&full_bar[stage]), phase, abort_flag)) { ok = false; break; }
                        tc_fence_after();
                        const uint32_t st = smem_u32(tiles + stage * kStageBytes);
                        const uint64_t dg = smem_desc_k128(st);
                        const uint64_t du = smem_desc_k128(st + kTileA);
                        const uint64_t db = smem_desc_k128(st + 2 * kTileA);
#pragma unroll
                        for (int kk = 0; kk < BK / UK; ++kk) {
                            // advance 16 elements = 32 bytes inside the swizzle atom
                            const uint64_t off = static_cast<uint64_t>((kk * UK * 2) >> 4);
                            const uint32_t acc = (kb > 0 || kk > 0) ? 1u : 0u;
                            umma_bf16(d_gate, dg + off, db + off, kIdesc, acc);
                            umma_bf16(d_up, du + off, db + off, kIdesc, acc);
                        }
                        umma_commit(smem_u32(&empty_bar[stage]));
                        if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                    }
                    if (!ok) break;
                    umma_commit(smem_u32(pass == 0 ? ab_full : acc_full));
                }
            }
            // Every MMA must have completed before TMEM is released.
            umma_commit(smem_u32(drain_bar));
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(smem_u32(drain_bar), 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;
        const int half = (warp - 2) >> 2;
        const int row = quad * 32 + lane;                 // neuron within the tile
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
        const uint32_t c0 = static_cast<uint32_t>(half * 64);
        uint32_t acc_phase = 0, ab_phase = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x) {
            // pass 0: convert (g, u) to (alpha, beta) in place
            if (!mbar_wait(smem_u32(ab_full), ab_phase, abort_flag)) { ok = false; break; }
            ab_phase ^= 1u;
            tc_fence_after();
#pragma unroll 1
            for (int i = 0; i < 4; ++i) {
                const uint32_t col = c0 + 16u * i;
                float g[16], uu[16];
                tmem_ld16(lane_base + kColAlpha + col, g);
                tmem_ld16(lane_base + kColBeta + col, uu);
                tmem_wait_ld();
                float a[16], b[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) swiglu_alpha_beta(g[e], uu[e], a[e], b[e]);
                tmem_st16(lane_base + kColAlpha + col, a);
                tmem_st16(lane_base + kColBeta + col, b);
            }
            tmem_wait_st();
            float* out = p.partial + (u * 2 + half) * static_cast<int64_t>(p.G) * BM;
            for (int h = 0; h < p.G; ++h) {
                if (!mbar_wait(smem_u32(acc_full), acc_phase, abort_flag)) { ok = false; break; }
                acc_phase ^= 1u;
                tc_fence_after();
                float pg[64], pu[64];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    tmem_ld16(lane_base + kColPg + c0 + 16u * i, &pg[16 * i]);
                    tmem_ld16(lane_base + kColPu + c0 + 16u * i, &pu[16 * i]);
                }
                tmem_wait_ld();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(acc_empty));
                float s = 0.0f;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float a[16], b[16];
                    tmem_ld16(lane_base + kColAlpha + c0 + 16u * i, a);
                    tmem_ld16(lane_base + kColBeta + c0 + 16u * i, b);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const float dlt = fmaf(a[e], pg[16 * i + e], b[e] * pu[16 * i + e]);
                        s = fmaf(dlt, dlt, s);
                    }
                }
                out[h * BM + row] = s;
            }
            if (!ok) break;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(ab_empty));
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

// A[h,k] += sum over token chunks (in order) of both column halves' partials.
__global__ void affinity_reduce_kernel(const float* __restrict__ partial, float* __restrict__ A, int G, int N,
                                       int NT, int TC) {
    const int64_t total = static_cast<int64_t>(G) * N;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int h = static_cast<int>(idx / N);
        const int k = static_cast<int>(idx % N);
        const int j = k / BM, r = k % BM;
        float sum = 0.0f;
        for (int c = 0; c < TC; ++c) {
            const int64_t base = ((static_cast<int64_t>(c) * NT + j) * 2) * G * BM + static_cast<int64_t>(h) * BM + r;
            sum += partial[base] + partial[base + static_cast<int64_t>(G) * BM];
        }
        A[idx] += sum;
    }
}

static PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
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

// bf16 tensor map with a [box_rows x 64] box and 128-byte swizzle; out-of-range
// elements read as zero, which contributes nothing to any sum below.
static bool make_map(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides,
                     cuuint32_t box_rows) {
    auto enc = get_encode_fn();
    if (!enc) return false;
    cuuint32_t box[3] = {static_cast<cuuint32_t>(BK), box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

size_t workspace_bytes(int64_t T, int d, int G, int N) {
    (void)d;
    const int64_t NT = (N + BM - 1) / BM;
    const int64_t TC = (T + BN - 1) / BN;
    return kWorkspaceHeader + static_cast<size_t>(NT * TC) * 2 * G * BM * sizeof(float);
}

int launch(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A,
           void* workspace, cudaStream_t stream) {
    CUtensorMap m_wg, m_wu, m_x, m_c;
    const cuuint64_t row_stride = static_cast<cuuint64_t>(d) * 2;
    cuuint64_t dw[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N)};
    cuuint64_t dx[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T)};
    cuuint64_t dc[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(G)};
    cuuint64_t s2[1] = {row_stride};
    cuuint64_t s3[2] = {row_stride, row_stride * static_cast<cuuint64_t>(T)};
    if (!make_map(&m_wg, Wg, 2, dw, s2, BM) || !make_map(&m_wu, Wu, 2, dw, s2, BM) ||
        !make_map(&m_x, X, 2, dx, s2, BN) || !make_map(&m_c, C, 3, dc, s3, BN))
        return DTP_ERR_CUDA;

    Params p;
    p.G = G;
    p.NT = (N + BM - 1) / BM;
    p.TC = static_cast<int>((T + BN - 1) / BN);
    p.KB = (d + BK - 1) / BK;
    p.units = static_cast<int64_t>(p.NT) * p.TC;
    p.status = reinterpret_cast<int*>(workspace);
    p.partial = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(workspace) + kWorkspaceHeader);

    int dev = 0, sms = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaFuncSetAttribute(affinity_fo_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBytes)));
    const int grid = static_cast<int>(p.units < sms ? p.units : sms);
    affinity_fo_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(m_wg, m_wu, m_x, m_c, p);
    DTP_CUDA_TRY(cudaGetLastError());
    const int64_t total = static_cast<int64_t>(G) * N;
    const int rblocks = static_cast<int>((total + 255) / 256 < 4 * sms ? (total + 255) / 256 : 4 * sms);
    affinity_reduce_kernel<<<rblocks, 256, 0, stream>>>(p.partial, A, G, N, p.NT, p.TC);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace tc
}  // namespace dtp
