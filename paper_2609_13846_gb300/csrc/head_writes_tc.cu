// head_writes_tc.cu -- the producer of the affinity pass's C (Sec. 3 "Affinity
// scores"): attention head h's write into the FFN input,
//
//     C[j, t, :] = gamma . (sum over heads h of row j of a_{h,t} W_o^(h)T) / r_t
//
// with a_h the head's output (columns h*hd .. of attn [T, Hq*hd]), W_o^(h) the
// matching columns of W_o [d, Hq*hd], gamma the FFN pre-norm gain and r_t the
// rms of the residual entering it.  Row j covers q_per_row consecutive heads,
// so j's columns are one contiguous range of length Kj = q_per_row * hd: one
// query head (q_per_row = 1) or one KV group's query heads.
//
// A GEMM with a short K (Kj = 96..512) whose output (T x d per row, bf16) is
// far larger than its inputs: the kernel is bound by the HBM write of C.
// Persistent grid, one CTA per SM, 20 warps.  Warp 0 loads 128 x 64 tiles of
// attn and 256 x 64 tiles of W_o by TMA, warp 1 issues 128 x 256 x 16
// tcgen05.mma into a double-buffered TMEM accumulator, and sixteen epilogue
// warps in two sets of eight drain it: set 0 takes the CTA's even units
// (TMEM buffer 0), set 1 the odd ones (buffer 1), so one set's TMEM loads and
// scaling overlap the other's stores.  An epilogue warp owns 32 tokens (its
// TMEM lane quadrant) x 128 columns and writes them as four 32 x 32 bf16
// boxes: scale by gamma / r in fp32 (packed f32x2 multiplies), round to bf16,
// store into a 64-byte-swizzled staging buffer and issue a TMA bulk store
// (two staging buffers per warp).  Boxes of 32 columns keep a thread's
// registers under the 102 that 640 threads allow.  Units are ordered with the
// 256-column tile fastest, so each 128-token tile of attn is read from HBM
// once and reused from L2 for every column tile.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace hw {

constexpr int BT = 128;       // tokens per tile (MMA M)
constexpr int BC = 256;       // output columns per tile (MMA N)
constexpr int BK = 64;
constexpr int UK = 16;
constexpr int STAGES = 3;
constexpr int kThreads = 640;
constexpr int kEpiWarps = 16;   // two sets of 8, one per TMEM buffer
constexpr int kEpiWarp0 = 4;
constexpr uint32_t kTileA = BT * BK * 2;          // 16 KB
constexpr uint32_t kTileB = BC * BK * 2;          // 32 KB
constexpr uint32_t kStageBytes = kTileA + kTileB;
constexpr uint32_t kStageOut = 32 * 64;           // one 32-row x 32-column bf16 box, 2 KB (64-byte swizzle)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBufCols = 256;
constexpr size_t kSmemBytes = 1024 + STAGES * kStageBytes + kEpiWarps * 2 * kStageOut + 256;
constexpr uint32_t kIdesc = idesc_bf16_f32(BT, BC);

struct Params {
    int rows;          // output rows j
    int TT;            // token tiles
    int DT;            // column tiles of 256
    int Kj;            // K of one row (multiple of 16)
    int KB;            // k blocks of 64
    int64_t units;     // rows * TT * DT
    int64_t T;
    int d;
    const float* gamma;
    const float* rms;
    int* status;
};

__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, uint32_t src, int32_t x, int32_t y, int32_t z) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(src), "r"(x), "r"(y), "r"(z)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Two fp32 products in one packed instruction (mul.rn.f32x2): each lane rounds as a scalar
// mul.rn.f32 does.
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(r.x), "=f"(r.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
}

// unit u -> (row j, token tile tt, column tile dc), column tile fastest
__device__ __forceinline__ void decode(const Params& p, int64_t u, int& j, int& tt, int& dc) {
    dc = static_cast<int>(u % p.DT);
    const int64_t q = u / p.DT;
    tt = static_cast<int>(q % p.TT);
    j = static_cast<int>(q / p.TT);
}

__global__ void __launch_bounds__(kThreads, 1)
head_writes_tc_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_w,
                      const __grid_constant__ CUtensorMap tm_c, const Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    uint8_t* staging = smem + STAGES * kStageBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(staging + kEpiWarps * 2 * kStageOut);
    uint64_t* full_bar = bars;
    uint64_t* empty_bar = bars + STAGES;
    uint64_t* acc_full = bars + 2 * STAGES;
    uint64_t* acc_empty = acc_full + 2;
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
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), kEpiWarps / 2);
        }
        mbar_init(smem_u32(drain_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tm_a);
        tma_prefetch_desc(&tm_w);
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

    if (warp == 0 && lane == 0) {
        // -------------------------------------------------------------------- producer
        int stage = 0;
        uint32_t phase = 0;
        uint32_t issued_parity[STAGES];
        bool issued[STAGES];
        for (int s = 0; s < STAGES; ++s) issued[s] = false, issued_parity[s] = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.units; u += gridDim.x) {
            int j, tt, dc;
            decode(p, u, j, tt, dc);
            for (int kb = 0; kb < p.KB; ++kb) {
                if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
                const uint32_t fb = smem_u32(&full_bar[stage]);
                uint8_t* st = tiles + stage * kStageBytes;
                const int x = j * p.Kj + kb * BK;       // 16-byte aligned: Kj and BK are multiples of 16
                mbar_arrive_expect_tx(fb, kStageBytes);
                tma_load_2d(smem_u32(st), &tm_a, fb, x, tt * BT);
                tma_load_2d(smem_u32(st + kTileA), &tm_w, fb, x, dc * BC);
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
                // the last block of a row may hold fewer than 64 of its columns (Kj = 96, ...):
                // only those enter the product; the rest of the tile belongs to the next row
                const int valid = p.Kj - kb * BK < BK ? p.Kj - kb * BK : BK;
                for (int kk = 0; kk < valid / UK; ++kk) {
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
        // set 0 takes the CTA's even units (TMEM buffer 0), set 1 the odd ones (buffer 1), so one
        // set's TMEM loads and scaling overlap the other's stores
        const int set = (warp - kEpiWarp0) >> 3;
        const int quad = warp & 3;                      // TMEM lanes 32*quad .. (tokens)
        const int half = ((warp - kEpiWarp0) >> 2) & 1; // columns 128*half .. of the tile
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
        uint8_t* stg = staging + (warp - kEpiWarp0) * 2 * kStageOut;
        uint32_t sbuf = 0;
        bool ok = true;
        const uint32_t buf = static_cast<uint32_t>(set);
        for (int64_t k = set;; k += 2) {
            const int64_t u = blockIdx.x + k * gridDim.x;
            if (!ok || u >= p.units) break;
            int j, tt, dc;
            decode(p, u, j, tt, dc);
            const uint32_t use = static_cast<uint32_t>((k >> 1) & 1);
            if (!mbar_wait(smem_u32(&acc_full[buf]), use, abort_flag)) { ok = false; break; }
            tc_fence_after();
            const int64_t t = static_cast<int64_t>(tt) * BT + quad * 32 + lane;
            const float rinv = t < p.T ? 1.0f / p.rms[t] : 0.0f;
            const float2 rr = make_float2(rinv, rinv);
            const int y0 = tt * BT + quad * 32;
            const uint32_t acc = lane_base + buf * kBufCols;
#pragma unroll 1
            for (int c = 0; c < 4; ++c) {
                const int col0 = 128 * half + 32 * c;
                const int g0 = dc * BC + col0;
                if (g0 >= p.d || y0 >= p.T) continue;   // box entirely outside C (warp-uniform)
                float4 gm[8];
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    gm[q] = g0 + 4 * q < p.d ? __ldg(reinterpret_cast<const float4*>(p.gamma + g0) + q)
                                             : make_float4(0.f, 0.f, 0.f, 0.f);
                float v[32];
                tmem_ld16(acc + static_cast<uint32_t>(col0), &v[0]);
                tmem_ld16(acc + static_cast<uint32_t>(col0 + 16), &v[16]);
                tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float2 s01 = mul2(make_float2(gm[q].x, gm[q].y), rr);
                    const float2 s23 = mul2(make_float2(gm[q].z, gm[q].w), rr);
                    const float2 a = mul2(make_float2(v[4 * q], v[4 * q + 1]), s01);
                    const float2 b = mul2(make_float2(v[4 * q + 2], v[4 * q + 3]), s23);
                    v[4 * q] = a.x; v[4 * q + 1] = a.y; v[4 * q + 2] = b.x; v[4 * q + 3] = b.y;
                }
                // the staging buffer is free once the store issued from it two boxes ago has read it
                if (lane == 0) bulk_wait_read1();
                __syncwarp();
                uint8_t* sb = stg + sbuf * kStageOut;
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    uint4 w;
                    w.x = pack_bf16(v[8 * cc], v[8 * cc + 1]);
                    w.y = pack_bf16(v[8 * cc + 2], v[8 * cc + 3]);
                    w.z = pack_bf16(v[8 * cc + 4], v[8 * cc + 5]);
                    w.w = pack_bf16(v[8 * cc + 6], v[8 * cc + 7]);
                    // 64-byte swizzle: 16-byte chunk cc of row `lane` sits at chunk cc ^ ((lane >> 1) & 3)
                    *reinterpret_cast<uint4*>(sb + lane * 64 + ((cc ^ ((lane >> 1) & 3)) << 4)) = w;
                }
                fence_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_3d(&tm_c, smem_u32(sb), g0, y0, j);
                    bulk_commit();
                }
                sbuf ^= 1u;
            }
            // its TMEM loads have completed (tcgen05.wait::ld): hand the buffer back without release
            // ordering, which would also wait for the warp's staging stores
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_relaxed(smem_u32(&acc_empty[buf]));
        }
        if (lane == 0) bulk_wait_all();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, static_cast<int>(DTP_ERR_NOT_CONVERGED));
}

static bool map_bf16(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides,
                     cuuint32_t box_x, cuuint32_t box_y, CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint32_t box[3] = {box_x, box_y, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// attn [T, Hq*hd], W_o [d, Hq*hd], C [Hq/q_per_row, T, d], all bf16; gamma [d], rms [T] fp32.
int launch(const void* attn, const void* Wo, const float* gamma, const float* rms, int64_t T, int d, int Hq, int hd,
           int q_per_row, void* C, void* workspace, cudaStream_t stream) {
    const int K = Hq * hd;
    const int rows = Hq / q_per_row;
    CUtensorMap ma, mw, mc;
    cuuint64_t da[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(T)};
    cuuint64_t dw[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(d)};
    cuuint64_t sk[1] = {static_cast<cuuint64_t>(K) * 2};
    cuuint64_t dc[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(rows)};
    cuuint64_t sc[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(d) * 2 * static_cast<cuuint64_t>(T)};
    if (!map_bf16(&ma, attn, 2, da, sk, BK, BT) || !map_bf16(&mw, Wo, 2, dw, sk, BK, BC) ||
        !map_bf16(&mc, C, 3, dc, sc, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B))
        return DTP_ERR_CUDA;
    Params p;
    p.rows = rows;
    p.TT = static_cast<int>((T + BT - 1) / BT);
    p.DT = (d + BC - 1) / BC;
    p.Kj = q_per_row * hd;
    p.KB = (p.Kj + BK - 1) / BK;
    p.units = static_cast<int64_t>(rows) * p.TT * p.DT;
    p.T = T;
    p.d = d;
    p.gamma = gamma;
    p.rms = rms;
    p.status = reinterpret_cast<int*>(workspace);
    int dev = 0, sms = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaFuncSetAttribute(head_writes_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBytes)));
    const int grid = static_cast<int>(p.units < sms ? p.units : sms);
    head_writes_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(ma, mw, mc, p);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace hw
}  // namespace dtp
