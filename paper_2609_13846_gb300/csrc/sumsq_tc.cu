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
// Structure as in affinity_tc.cu, with the same two forms: CTA pairs sharing
// one 256 x 256 x 16 tcgen05.mma of cta_group::2 per K step (each CTA stages
// its 128 rows of A and half of B -- 128 of the 256 columns for the down edge,
// the W_gate rows in the even CTA and the W_up rows in the odd one for ADD --
// in three stages of 128 k columns) when B fits in half of L2, else single
// CTAs with one 128 x 256 x 16 tcgen05.mma per K step and four 64-wide stages.
// Persistent grid, one CTA per SM, warp 0 TMA producer, warp 1 MMA issuer,
// eight epilogue warps; TMEM double-buffered across units.  A unit is (row
// group, row chunk -- a pair of row chunks in the pair form --, column tile).
// The epilogue sums the squares over its warp's 32 rows with a shuffle
// butterfly and over the four lane quadrants in shared memory in a fixed
// order; each chunk writes its own partial slot and a reduce kernel adds the
// row chunks in order, so the result is deterministic.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "dtp_common.cuh"

namespace dtp {
namespace sq {

constexpr int BR = 128;       // rows per chunk (MMA M, TMEM lanes)
constexpr int BCOL = 256;     // MMA N
constexpr int BK = 64;
constexpr int UK = 16;
constexpr int kThreads = 384;
constexpr int kEpiWarps = 8;
constexpr int kEpiWarp0 = 4;
constexpr uint32_t kTileA = BR * BK * 2;          // 16 KB
constexpr uint32_t kTileB = BCOL * BK * 2;        // 32 KB (both halves of B)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBufCols = 256;
constexpr size_t kRedBytes = 2 * 4 * BCOL * sizeof(float);   // [slot][quadrant][column]

// Per form (as in affinity_tc.cu): a stage holds kBoxes 64-wide k blocks of A and of B (half of
// B in the pair form); both forms keep 192 KB of stages in flight.
template <bool kPair>
struct Form {
    static constexpr int kBoxes = kPair ? 2 : 1;
    static constexpr uint32_t kBoxBytes = kTileA + (kPair ? kTileB / 2 : kTileB);
    static constexpr int STAGES = kPair ? 3 : 4;
    static constexpr uint32_t kStageBytes = kBoxes * kBoxBytes;
    static constexpr uint32_t kIdesc = idesc_bf16_f32(kPair ? 2 * BR : BR, BCOL);
    static constexpr size_t kSmemBytes = 1024 + STAGES * kStageBytes + kRedBytes + 256;
};
static_assert(Form<true>::kSmemBytes <= 227 * 1024 && Form<false>::kSmemBytes <= 227 * 1024, "shared memory");

enum Mode { kDown = 0, kAdd = 1 };

struct Params {
    int groups;       // row groups (KV groups)
    int row_chunks;   // chunks of 128 rows per group
    int rc_slots;     // partial slots per group: row_chunks rounded up to an even count
    int row_units;    // row chunks per unit: pairs ceil(row_chunks / 2) (pair form) or row_chunks
    int col_tiles;    // column tiles
    int KB;           // k blocks of 64
    int KS;           // stages per unit, ceil(KB / kBoxes)
    int64_t units;    // groups * row_units * col_tiles
    int out_cols;     // outputs per unit: 256 (kDown) or 128 (kAdd)
    float* partial;   // [groups][rc_slots][col_tiles][out_cols]
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

// unit u -> (group, row unit, column tile), column tile fastest so a row chunk
// stays in L2 while it meets every column tile
__device__ __forceinline__ void decode(const Params& p, int64_t u, int& g, int& ru, int& j) {
    j = static_cast<int>(u % p.col_tiles);
    const int64_t q = u / p.col_tiles;
    ru = static_cast<int>(q % p.row_units);
    g = static_cast<int>(q / p.row_units);
}

template <int MODE, bool kPair>
__global__ void __launch_bounds__(kThreads, 1)
sumsq_tc_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b0,
                const __grid_constant__ CUtensorMap tm_b1, const Params p) {
    constexpr int STAGES = Form<kPair>::STAGES;
    constexpr int kBoxes = Form<kPair>::kBoxes;
    constexpr uint32_t kBoxBytes = Form<kPair>::kBoxBytes;
    constexpr uint32_t kStageBytes = Form<kPair>::kStageBytes;
    constexpr uint32_t kIdesc = Form<kPair>::kIdesc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    float* red = reinterpret_cast<float*>(smem + STAGES * kStageBytes);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * kStageBytes + kRedBytes);
    // full[S], empty[S], acc_full[2], acc_empty[2], red_full[2], drain.  In the pair form full and
    // acc_empty are used in the even CTA only; empty, acc_full and drain receive its commits in both.
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
    const uint32_t rank = kPair ? cluster_ctarank() : 0u;   // 0: issues the MMAs; 1: its peer
    const bool leader = rank == 0;
    const int64_t worker = kPair ? blockIdx.x >> 1 : blockIdx.x;
    const int64_t workers = kPair ? gridDim.x >> 1 : gridDim.x;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), (kPair ? 2 : 1) * kEpiWarps);
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
        if constexpr (kPair) {
            tmem_alloc_pair(smem_u32(tmem_slot), kTmemCols);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(smem_u32(tmem_slot), kTmemCols);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    if constexpr (kPair)
        cluster_sync();   // both CTAs' barriers initialised and TMEM allocated before any remote access
    else
        __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // -------------------------------------------------------------------- producer
        const uint32_t full_lead = kPair ? mapa_shared(smem_u32(full_bar), 0) : 0u;
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int64_t u = worker; ok && u < p.units; u += workers) {
            int g, ru, j;
            decode(p, u, g, ru, j);
            // the odd CTA of a last, half-empty pair reloads the last chunk (its sums go to a spare slot)
            const int rc_raw = kPair ? 2 * ru + static_cast<int>(rank) : ru;
            const int rc = rc_raw < p.row_chunks ? rc_raw : p.row_chunks - 1;
            for (int ks = 0; ks < p.KS; ++ks) {
                if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
                const uint32_t st = smem_u32(tiles + stage * kStageBytes);
                const uint32_t fb = kPair ? full_lead + static_cast<uint32_t>(stage) * 8u : smem_u32(&full_bar[stage]);
                auto load_box = [&](int hb, int x) {
                    const uint32_t sb = st + hb * kBoxBytes;
                    if constexpr (kPair) {
                        tma_load_3d_pair(sb, &tm_a, fb, x, rc * BR, g);
                        if (MODE == kDown)
                            tma_load_2d_pair(sb + kTileA, &tm_b0, fb, x, j * BCOL + static_cast<int>(rank) * (BCOL / 2));
                        else
                            tma_load_2d_pair(sb + kTileA, leader ? &tm_b0 : &tm_b1, fb, x, j * (BCOL / 2));
                    } else {
                        tma_load_3d(sb, &tm_a, fb, x, rc * BR, g);
                        if (MODE == kDown) {
                            tma_load_2d(sb + kTileA, &tm_b0, fb, x, j * BCOL);
                        } else {
                            tma_load_2d(sb + kTileA, &tm_b0, fb, x, j * (BCOL / 2));
                            tma_load_2d(sb + kTileA + kTileB / 2, &tm_b1, fb, x, j * (BCOL / 2));
                        }
                    }
                };
                if constexpr (kBoxes == 1) {
                    if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[stage]), (kPair ? 2u : 1u) * kStageBytes);
                    load_box(0, ks * BK);
                } else {
                    // k blocks in this stage: kBoxes, fewer in the last stage when KB is odd
                    const int nb = p.KB - ks * kBoxes < kBoxes ? p.KB - ks * kBoxes : kBoxes;
                    if (leader)
                        mbar_arrive_expect_tx(smem_u32(&full_bar[stage]),
                                              (kPair ? 2u : 1u) * static_cast<uint32_t>(nb) * kBoxBytes);
                    if (nb == kBoxes) {
#pragma unroll
                        for (int hb = 0; hb < kBoxes; ++hb) load_box(hb, (ks * kBoxes + hb) * BK);
                    } else {
                        for (int hb = 0; hb < nb; ++hb) load_box(hb, (ks * kBoxes + hb) * BK);
                    }
                }
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
        }
    } else if (warp == 1 && lane == 0 && leader) {
        // ------------------------------------------------------------------ MMA issuer (the even CTA of a pair)
        int stage = 0;
        uint32_t phase = 0, unit_count = 0;
        bool ok = true;
        for (int64_t u = worker; ok && u < p.units; u += workers, ++unit_count) {
            const uint32_t buf = unit_count & 1u;
            const uint32_t use = (unit_count >> 1) & 1u;
            const bool freed = kPair ? mbar_wait_cluster(smem_u32(&acc_empty[buf]), use ^ 1u, abort_flag)
                                     : mbar_wait(smem_u32(&acc_empty[buf]), use ^ 1u, abort_flag);
            if (!freed) { ok = false; break; }
            tc_fence_after();
            const uint32_t d_acc = tmem + buf * kBufCols;
            for (int ks = 0; ks < p.KS; ++ks) {
                const bool landed = kPair ? mbar_wait_cluster(smem_u32(&full_bar[stage]), phase, abort_flag)
                                          : mbar_wait(smem_u32(&full_bar[stage]), phase, abort_flag);
                if (!landed) { ok = false; break; }
                tc_fence_after();
                const uint32_t st = smem_u32(tiles + stage * kStageBytes);
                auto mma_box = [&](int hb, bool first) {
                    const uint64_t da = smem_desc_k128(st + hb * kBoxBytes);
                    const uint64_t db = smem_desc_k128(st + hb * kBoxBytes + kTileA);
#pragma unroll
                    for (int kk = 0; kk < BK / UK; ++kk) {
                        const uint64_t off = static_cast<uint64_t>((kk * UK * 2) >> 4);
                        const uint32_t accumulate = (first && kk == 0) ? 0u : 1u;
                        if constexpr (kPair)
                            umma_bf16_pair(d_acc, da + off, db + off, kIdesc, accumulate);
                        else
                            umma_bf16(d_acc, da + off, db + off, kIdesc, accumulate);
                    }
                };
                if constexpr (kBoxes == 1) {
                    mma_box(0, ks == 0);
                } else {
                    const int nb = p.KB - ks * kBoxes < kBoxes ? p.KB - ks * kBoxes : kBoxes;
                    if (nb == kBoxes) {
#pragma unroll
                        for (int hb = 0; hb < kBoxes; ++hb) mma_box(hb, ks == 0 && hb == 0);
                    } else {
                        for (int hb = 0; hb < nb; ++hb) mma_box(hb, ks == 0 && hb == 0);
                    }
                }
                if constexpr (kPair)
                    umma_commit_pair(smem_u32(&empty_bar[stage]), 3);
                else
                    umma_commit(smem_u32(&empty_bar[stage]));
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
            if (!ok) break;
            if constexpr (kPair)
                umma_commit_pair(smem_u32(&acc_full[buf]), 3);
            else
                umma_commit(smem_u32(&acc_full[buf]));
        }
        // Every MMA must have completed before TMEM or shared memory is released.
        if constexpr (kPair)
            umma_commit_pair(smem_u32(drain_bar), 3);
        else
            umma_commit(smem_u32(drain_bar));
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
        // release of an accumulator buffer: in the pair form an arrival on the even CTA's barrier
        auto release = [&](uint32_t buf) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if constexpr (kPair)
                    mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(&acc_empty[buf]), 0));
                else
                    mbar_arrive(smem_u32(&acc_empty[buf]));
            }
        };
        uint32_t unit_count = 0;
        bool ok = true;
        for (int64_t u = worker; ok && u < p.units; u += workers, ++unit_count) {
            int g, ru, j;
            decode(p, u, g, ru, j);
            // row chunk rc = row_chunks (the empty half of a last pair) writes a spare slot
            const int rc = kPair ? 2 * ru + static_cast<int>(rank) : ru;
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
            if (!summer) release(buf);
#pragma unroll
            for (int blk = 0; blk < kBlocks; ++blk) rs[quad * BCOL + kPerHalf * half + 32 * blk + lane] = colsum[blk];
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&red_full[slot]));
            if (summer) {
                if (!mbar_wait(smem_u32(&red_full[slot]), rphase, abort_flag)) { ok = false; break; }
                const int64_t slot_idx = (static_cast<int64_t>(g) * p.rc_slots + rc) * p.col_tiles + j;
                float* o = p.partial + slot_idx * p.out_cols + kPerHalf * half;
#pragma unroll
                for (int blk = 0; blk < kBlocks; ++blk) {
                    const int n = kPerHalf * half + 32 * blk + lane;
                    o[32 * blk + lane] = ((rs[n] + rs[BCOL + n]) + rs[2 * BCOL + n]) + rs[3 * BCOL + n];
                }
                // only now may the buffer (and, two units later, this red slot) be reused
                release(buf);
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1 && lane == 0) {
        // the last MMA commit: every MMA (in the pair form reading both CTAs' tiles and writing
        // both CTAs' TMEM) has completed
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(smem_u32(drain_bar), 0) && globaltimer_ns() - t0 < kWaitLimitNs) {
        }
    }
    // After a wait gave up, loads already issued (in the pair form also the peer's) may still be
    // landing in this CTA's shared memory or on its barriers: let them finish before exiting.
    if constexpr (kPair) {
        cluster_sync();
        if (threadIdx.x == 0) {
            const int peer_abort = static_cast<int>(ld_shared_cluster_u32(
                mapa_shared(smem_u32(const_cast<int*>(abort_flag)), rank ^ 1u)));
            if (*abort_flag || peer_abort) {
                const uint64_t t0 = globaltimer_ns();
                while (globaltimer_ns() - t0 < 200ull * 1000ull) {
                }
            }
        }
        cluster_sync();
    } else {
        if (threadIdx.x == 0 && *abort_flag) {
            const uint64_t t0 = globaltimer_ns();
            while (globaltimer_ns() - t0 < 200ull * 1000ull) {
            }
        }
        __syncthreads();
    }
    if (warp == 1) {
        tc_fence_after();
        if constexpr (kPair)
            tmem_dealloc_pair(tmem, kTmemCols);
        else
            tmem_dealloc(tmem, kTmemCols);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicExch(p.status, static_cast<int>(DTP_ERR_NOT_CONVERGED));
}

// out[g, col] (+)= sum over row chunks (in order) of the unit partials; col < n_cols.
// out row o sums groups o*qpg .. o*qpg + qpg - 1 (group by group, then row chunks); a group's
// partials occupy rc_slots >= row_chunks slots (the spare ones are never read).
__global__ void sumsq_reduce_kernel(const float* __restrict__ partial, float* __restrict__ out, int groups,
                                    int row_chunks, int rc_slots, int col_tiles, int out_cols, int n_cols,
                                    int accumulate, int qpg) {
    const int64_t total = static_cast<int64_t>(groups / qpg) * n_cols;
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int o = static_cast<int>(idx / n_cols);
        const int col = static_cast<int>(idx % n_cols);
        const int j = col / out_cols, r = col % out_cols;
        float s = 0.0f;
        for (int g = o * qpg; g < (o + 1) * qpg; ++g)
            for (int rc = 0; rc < row_chunks; ++rc)
                s += partial[((static_cast<int64_t>(g) * rc_slots + rc) * col_tiles + j) * out_cols + r];
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

static bool map_bf16(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides,
                     cuuint32_t box_rows) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint32_t box[3] = {static_cast<cuuint32_t>(BK), box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Fills the form-dependent fields of p (row_units, KS, units), launches the main kernel (CTA pairs
// when B, b_bytes in all, fits in half of L2 and a cluster of two can be resident) and the reduce.  mb0p / mb1p are B's maps for the pair
// form (boxes of 128 rows), mb0 / mb1 for the single form.
template <int MODE>
static int run(const CUtensorMap& ma, const CUtensorMap& mb0, const CUtensorMap& mb1, const CUtensorMap& mb0p,
               const CUtensorMap& mb1p, double b_bytes, Params p, float* out, int n_cols, int accumulate,
               cudaStream_t stream, int qpg = 1) {
    int dev = 0, sms = 0, l2 = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev));
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.stream = stream;
    cfg.attrs = attr;
    // CTA pairs resident at once, queried once per device and mode (0: not yet; -1: none can be,
    // and the single form runs instead)
    int resident = 0;
    if (b_bytes <= l2 / 2.0) {
        static std::atomic<int> resident_cache[2][64];
        resident = dev < 64 ? resident_cache[MODE][dev].load(std::memory_order_relaxed) : 0;
        if (resident == 0) {
            DTP_CUDA_TRY(cudaFuncSetAttribute(sumsq_tc_kernel<MODE, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(Form<true>::kSmemBytes)));
            cfg.gridDim = dim3(static_cast<unsigned>(sms & ~1), 1, 1);
            cfg.dynamicSmemBytes = Form<true>::kSmemBytes;
            cfg.numAttrs = 1;
            if (cudaOccupancyMaxActiveClusters(&resident, sumsq_tc_kernel<MODE, true>, &cfg) != cudaSuccess ||
                resident < 1) {
                (void)cudaGetLastError();
                resident = -1;
            }
            if (dev < 64) resident_cache[MODE][dev].store(resident, std::memory_order_relaxed);
        }
    }
    const bool pair = resident > 0;
    auto kernel = pair ? sumsq_tc_kernel<MODE, true> : sumsq_tc_kernel<MODE, false>;
    const size_t smem = pair ? Form<true>::kSmemBytes : Form<false>::kSmemBytes;
    DTP_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
    attr[0].val.clusterDim.x = pair ? 2 : 1;
    cfg.dynamicSmemBytes = smem;
    cfg.numAttrs = pair ? 1 : 0;
    int workers;
    if (pair) {
        p.row_units = (p.row_chunks + 1) / 2;
        p.KS = (p.KB + Form<true>::kBoxes - 1) / Form<true>::kBoxes;
        workers = sms / 2 < resident ? sms / 2 : resident;
    } else {
        p.row_units = p.row_chunks;
        p.KS = (p.KB + Form<false>::kBoxes - 1) / Form<false>::kBoxes;
        workers = sms;
    }
    p.units = static_cast<int64_t>(p.groups) * p.row_units * p.col_tiles;
    if (p.units < workers) workers = static_cast<int>(p.units);
    if (workers < 1) workers = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(pair ? 2 * workers : workers), 1, 1);
    if (pair)
        DTP_CUDA_TRY(cudaLaunchKernelEx(&cfg, kernel, ma, mb0p, mb1p, p));
    else
        DTP_CUDA_TRY(cudaLaunchKernelEx(&cfg, kernel, ma, mb0, mb1, p));
    DTP_CUDA_TRY(cudaGetLastError());
    const int64_t total = static_cast<int64_t>(p.groups / qpg) * n_cols;
    const int blocks = static_cast<int>((total + 255) / 256 < 4 * sms ? (total + 255) / 256 : 4 * sms);
    sumsq_reduce_kernel<<<blocks, 256, 0, stream>>>(p.partial, out, p.groups, p.row_chunks, p.rc_slots, p.col_tiles,
                                                    p.out_cols, n_cols, accumulate, qpg);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

// ---------------------------------------------------------------- down edge --

// partial slots per group: the row-chunk count rounded up to an even count
static int64_t rc_slots(int64_t rows) { return ((rows + BR - 1) / BR + 1) / 2 * 2; }

size_t down_workspace_bytes(int G, int R, int d, int N) {
    const int64_t units = static_cast<int64_t>(G) * rc_slots(R) * ((N + BCOL - 1) / BCOL);
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
    CUtensorMap ma, mb, mbp;
    const cuuint64_t rs = static_cast<cuuint64_t>(d) * 2;
    cuuint64_t da[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(R), static_cast<cuuint64_t>(G)};
    cuuint64_t sa[2] = {rs, rs * static_cast<cuuint64_t>(R)};
    cuuint64_t db[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N)};
    cuuint64_t sb[1] = {rs};
    if (!map_bf16(&ma, Wqkv, 3, da, sa, BR) || !map_bf16(&mb, WdT, 2, db, sb, BCOL) ||
        !map_bf16(&mbp, WdT, 2, db, sb, BCOL / 2))
        return DTP_ERR_CUDA;
    Params p;
    p.groups = G;
    p.row_chunks = (R + BR - 1) / BR;
    p.rc_slots = static_cast<int>(rc_slots(R));
    p.col_tiles = (N + BCOL - 1) / BCOL;
    p.KB = (d + BK - 1) / BK;
    p.out_cols = BCOL;
    p.partial = partial;
    p.status = reinterpret_cast<int*>(ws);
    return run<kDown>(ma, mb, mb, mbp, mbp, static_cast<double>(N) * d * 2, p, bn, N, 0, stream);
}

// ---------------------------------------------------------------- ADD score --

size_t add_workspace_bytes(int64_t T, int G, int N) {
    const int64_t units = static_cast<int64_t>(G) * rc_slots(T) * ((N + 127) / 128);
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
    p.rc_slots = static_cast<int>(rc_slots(T));
    p.col_tiles = (N + 127) / 128;
    p.KB = (d + BK - 1) / BK;
    p.out_cols = 128;
    p.partial = reinterpret_cast<float*>(ws + kWorkspaceHeader);
    p.status = reinterpret_cast<int*>(ws);
    // the gate and up maps already have boxes of 128 rows: the same maps serve both forms
    return run<kAdd>(mc, mg, mu, mg, mu, 2.0 * N * d * 2, p, A_add, N, 1, stream, qpg);
}

int launch_add(const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A_add,
               void* workspace, cudaStream_t stream) {
    return launch_add_grouped(C, Wg, Wu, T, d, G, N, A_add, workspace, stream, 1);
}

}  // namespace sq
}  // namespace dtp
