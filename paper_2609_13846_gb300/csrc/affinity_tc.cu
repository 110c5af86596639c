// affinity_tc.cu -- first-order head->neuron affinity on the tcgen05 tensor
// cores (bf16 operands, fp32 accumulation), Sec. 3 "Affinity scores":
//
//     A[h,k] += sum_t ( silu'(g_tk) u_tk pg_thk + silu(g_tk) pu_thk )^2
//
// with g = X W_gate^T, u = X W_up^T (the operating point) and pg = C_h W_gate^T,
// pu = C_h W_up^T (head h's piece projected through the FFN input weights).
//
// MMA shape, two forms of one kernel (template parameter kPair):
//  - CTA pairs (clusters of two) sharing one tcgen05.mma of cta_group::2 per
//    16-wide K step: M = 256 tokens (128 token rows of one activation tile,
//    X or C_h, in each CTA), N = 256 columns (the neuron tile's 128 W_gate
//    rows in the even CTA, its 128 W_up rows in the odd CTA).  Each SM stages
//    and reads only half of the weight operand, which keeps the tensor pipe
//    busier than a single-CTA instruction does.  Used when the weights fit in
//    L2 with room to spare.
//  - single CTAs issuing one tcgen05.mma of cta_group::1 per K step: M = 128
//    tokens, N = 256 (W_gate and W_up tiles stacked).  Used for layers whose
//    weights do not fit in L2: there the pairs' placement (a cluster's CTAs
//    land on neighbouring SMs, consecutive clusters fill one part of the chip
//    after another) cost the chunk grouping below most of its L2 reuse --
//    several times the DRAM traffic on a Llama-3.1-8B-shaped layer.
// In both, columns [0,128) of a CTA's accumulator are g (or pg) and [128,256)
// are u (or pu) of the same 128 neurons for that CTA's 128 tokens.
//
// Work unit = (chunk unit, neuron tile j of 128 neurons); a chunk unit is a
// pair of 128-token chunks (2 cu for the even CTA, 2 cu + 1 for the odd one)
// in the pair form and one chunk in the single form.  A unit runs G+1 passes
// over d: pass 0 multiplies the X chunks, pass 1+h the C_h chunks.  Units are
// dealt round-robin to a persistent grid in chunk-unit-major order, so the
// units in flight share a handful of token chunks in L2 while all weights
// stay L2-resident.  When the weights do not fit in L2, chunk units are taken
// in groups and each neuron tile meets the group's chunk units back to back,
// so the units in flight share fewer weight tiles.  The units left over after
// the last full round are split by heads over several workers (each
// recomputes the unit's X pass), so the final round keeps most SMs busy.  In
// the pair form with an odd chunk count, the odd CTA of the last pair reloads
// the last chunk and stores its sums into a spare slot the reduce never reads.
//
// Pair protocol.  Both CTAs' TMA loads of a stage complete on the even CTA's
// full barrier (one expect-tx of both CTAs' bytes); the even CTA's single MMA
// thread waits there, issues the pair MMAs and commits to the empty barriers
// and accumulator barriers of both CTAs at once (multicast); the epilogue
// warps of both CTAs release an accumulator buffer by arriving on the even
// CTA's barrier.
//
// TMEM (512 columns x 128 lanes = tokens, fp32): two accumulator buffers of
// 256 columns used by passes alternately, so the epilogue of one pass
// overlaps the MMAs of the next.
//
// Epilogue.  Two warps per TMEM lane quadrant (32 tokens) split the 128
// neurons into halves of 64.  A warp reads its accumulator with 16-lane loads
// (tcgen05.ld 16x256b), so each thread owns 4 tokens x 16 neurons.  Pass 0
// leaves alpha = silu'(g) u and beta = silu(g) of the thread's 64 (token,
// neuron) pairs in registers for the whole unit.  A head pass forms Delta^2 for
// the same pairs, sums it over the thread's 4 tokens (fused multiply-adds),
// then over the 8 lanes sharing its neurons (a 3-round shuffle butterfly), and
// the four quadrant warps' sums are added in shared memory in a fixed order.
// The T x G x N intermediate never leaves the SM; each unit writes its G x 128
// partial sums to its own workspace slot and a second kernel adds them into A
// in a fixed order, so the result is deterministic.
//
// Down-edge activation term (optional): with the rms r' of the residual that
// enters the next layer's pre-norm, the X pass also sums (silu(g) u)^2 / r'^2
// over tokens per neuron -- E_t[alpha_k^2 / r'^2] of the down-edge score before
// the mean -- with the same butterfly and quadrant reduction.
//
// Warp roles (384 threads, 3 warpgroups per CTA): warp 0 issues TMA loads,
// warp 1 allocates TMEM (for the pair in the pair form) and issues the MMAs
// (one thread; in the pair form only in the even CTA), warps 2-3 idle;
// warpgroup 0 gives registers back (setmaxnreg) to warpgroups 1-2, the
// epilogue.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "dtp_common.cuh"

namespace dtp {
namespace tc {

constexpr int BT = 128;       // tokens per chunk (MMA M, TMEM lanes)
constexpr int BNEU = 128;     // neurons per tile (MMA N = 2 * BNEU: gate | up)
constexpr int BK = 64;        // bf16 elements per 128-byte swizzled row
constexpr int UK = 16;        // K of one tcgen05.mma kind::f16
constexpr int kThreads = 384;
constexpr int kEpiWarps = 8;
constexpr int kEpiWarp0 = 4;  // first epilogue warp
constexpr uint32_t kRegsSmall = 56;   // warpgroup 0 after setmaxnreg.dec
constexpr uint32_t kRegsLarge = 224;  // epilogue warpgroups after setmaxnreg.inc
static_assert(128 * kRegsSmall + 256 * kRegsLarge <= kThreads * 168, "register split exceeds the launch budget");
constexpr uint32_t kTileAct = BT * BK * 2;     // 16 KB activation operand (this CTA's A rows)
constexpr uint32_t kTileW = BNEU * BK * 2;     // 16 KB: the W_gate or the W_up rows of a neuron tile
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBufCols = 256;
constexpr size_t kRedBytes = 2 * 4 * BNEU * sizeof(float);   // [slot][quadrant][neuron]

// Per form: a stage holds kBoxes 64-wide k blocks, each this CTA's activation box and its weight
// box(es) (half of B in the pair form, both halves in the single form); both forms keep 192 KB of
// stages in flight.  The pair form takes 128 k columns per stage: its MMA thread then waits on a
// barrier once per eight MMAs instead of four, which measured ~7% faster than six 64-wide stages.
template <bool kPair>
struct Form {
    static constexpr int kBoxes = kPair ? 2 : 1;
    static constexpr uint32_t kBoxBytes = kTileAct + (kPair ? 1u : 2u) * kTileW;
    static constexpr int STAGES = kPair ? 3 : 4;
    static constexpr uint32_t kStageBytes = kBoxes * kBoxBytes;
    static constexpr uint32_t kIdesc = idesc_bf16_f32(kPair ? 2 * BT : BT, 2 * BNEU);
    static constexpr size_t kSmemBytes = 1024 + STAGES * kStageBytes + kRedBytes + 256;
};
static_assert(Form<true>::kSmemBytes <= 227 * 1024 && Form<false>::kSmemBytes <= 227 * 1024, "shared memory");

struct Params {
    int G;            // KV heads
    int NT;           // neuron tiles
    int TC;           // token chunks
    int TU;           // chunk units: chunk pairs ceil(TC / 2) (pair form) or chunks (single form)
    int KB;           // k blocks of 64 over d
    int KS;           // stages per pass, ceil(KB / kBoxes)
    int64_t units;    // NT * TU
    int full_rounds;  // rounds in which every worker (CTA pair or CTA) takes one whole unit
    int split;        // head groups per left-over unit
    int tail_items;   // left-over units * split (<= workers)
    int cg;           // chunk units per group of the unit order (1 = chunk-unit-major)
    int64_t T;        // tokens
    float* partial;   // [units][G][128]
    const float* rms; // [T] rms of the next layer's pre-norm input, or null
    float* partial_act;  // [units][128] down-edge activation sums (when rms is set)
    int* status;      // workspace status word
};

// The i-th work item of a worker (a CTA pair or a CTA): a unit and the head range [h0, h1) it covers.
struct Item {
    int64_t unit;
    int h0, h1;
};

// Unit u in the processing order -> (chunk unit cu, neuron tile j).  The chunk of a CTA is
// 2 cu + (its rank in the pair) in the pair form and cu in the single form.
__device__ __forceinline__ void unit_coords(const Params& p, int64_t u, int& cu, int& j) {
    const int64_t per_group = static_cast<int64_t>(p.cg) * p.NT;
    const int64_t grp = u / per_group;
    const int64_t r = u - grp * per_group;
    const int c0 = static_cast<int>(grp) * p.cg;
    const int cn = p.TU - c0 < p.cg ? p.TU - c0 : p.cg;   // chunk units in this (possibly last) group
    j = static_cast<int>(r / cn);
    cu = c0 + static_cast<int>(r % cn);
}

// Workers: CTA pairs (clusters of two, blocks 2q and 2q + 1 form pair q) or single CTAs.
template <bool kPair>
__device__ __forceinline__ bool get_item(const Params& p, int i, Item& it) {
    const int worker = static_cast<int>(kPair ? blockIdx.x >> 1 : blockIdx.x);
    const int workers = static_cast<int>(kPair ? gridDim.x >> 1 : gridDim.x);
    if (i < p.full_rounds) {
        it.unit = static_cast<int64_t>(i) * workers + worker;
        it.h0 = 0;
        it.h1 = p.G;
        return true;
    }
    if (i == p.full_rounds && worker < p.tail_items) {
        const int t = worker;
        const int grp = t % p.split;
        it.unit = static_cast<int64_t>(p.full_rounds) * workers + t / p.split;
        it.h0 = p.G * grp / p.split;
        it.h1 = p.G * (grp + 1) / p.split;
        return true;
    }
    return false;
}

template <bool kPair>
__global__ void __launch_bounds__(kThreads, 1)
affinity_fo_tc_kernel(const __grid_constant__ CUtensorMap tm_wg, const __grid_constant__ CUtensorMap tm_wu,
                      const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_c,
                      const Params p) {
    constexpr int STAGES = Form<kPair>::STAGES;
    constexpr int kBoxes = Form<kPair>::kBoxes;
    constexpr uint32_t kBoxBytes = Form<kPair>::kBoxBytes;
    constexpr uint32_t kStageBytes = Form<kPair>::kStageBytes;
    constexpr uint32_t kIdesc = Form<kPair>::kIdesc;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* tiles = smem;
    float* red = reinterpret_cast<float*>(smem + STAGES * kStageBytes);   // [2][4][128]
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * kStageBytes + kRedBytes);
    // full[S], empty[S], acc_full[2], acc_empty[2], red_full[2], red_empty[2], drain.  In the pair
    // form full and acc_empty are used in the even CTA only (both CTAs' loads and epilogues arrive
    // there); empty, acc_full and drain receive the even CTA's commits in both CTAs.
    uint64_t* full_bar = bars;
    uint64_t* empty_bar = bars + STAGES;
    uint64_t* acc_full = bars + 2 * STAGES;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* red_full = acc_full + 4;
    uint64_t* red_empty = acc_full + 6;
    uint64_t* drain_bar = acc_full + 8;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_full + 9);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = kPair ? cluster_ctarank() : 0u;   // 0: issues the MMAs; 1: its peer
    const bool leader = rank == 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&full_bar[s]), 1);
            mbar_init(smem_u32(&empty_bar[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&acc_full[b]), 1);
            mbar_init(smem_u32(&acc_empty[b]), (kPair ? 2 : 1) * kEpiWarps);
            mbar_init(smem_u32(&red_full[b]), kEpiWarps);
            mbar_init(smem_u32(&red_empty[b]), 2);   // the two summing warps
        }
        mbar_init(smem_u32(drain_bar), 1);
        *abort_flag = 0;
        fence_mbar_init();
        if (!kPair || leader) tma_prefetch_desc(&tm_wg);
        if (!kPair || !leader) tma_prefetch_desc(&tm_wu);
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_c);
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

    if (warp < kEpiWarp0) {
        setmaxnreg_dec<kRegsSmall>();
        if (warp == 0 && lane == 0) {
            // ---------------------------------------------------------------- producer (every CTA)
            const uint32_t full_lead = kPair ? mapa_shared(smem_u32(full_bar), 0) : 0u;   // the even CTA's full[0]
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            Item it;
            for (int i = 0; ok && get_item<kPair>(p, i, it); ++i) {
                int cu, j;
                unit_coords(p, it.unit, cu, j);
                // the odd CTA of a last, half-empty pair reloads the last chunk (its sums go to a spare slot)
                const int c_raw = kPair ? 2 * cu + static_cast<int>(rank) : cu;
                const int c = c_raw < p.TC ? c_raw : p.TC - 1;
                const int passes = 1 + it.h1 - it.h0;
                for (int pass = 0; ok && pass < passes; ++pass) {
                    for (int ks = 0; ks < p.KS; ++ks) {
                        if (!mbar_wait(smem_u32(&empty_bar[stage]), phase ^ 1u, abort_flag)) { ok = false; break; }
                        // k blocks in this stage: kBoxes, fewer in a pass's last stage when KB is odd
                        const int nb = kBoxes == 1 ? 1 : (p.KB - ks * kBoxes < kBoxes ? p.KB - ks * kBoxes : kBoxes);
                        const uint32_t st = smem_u32(tiles + stage * kStageBytes);
                        // loads of k block x0 / BK into box hb of the stage
                        auto load_box = [&](int hb, uint32_t fb, int x) {
                            const uint32_t sb = st + hb * kBoxBytes;
                            if constexpr (kPair) {
                                if (pass == 0)
                                    tma_load_2d_pair(sb, &tm_x, fb, x, c * BT);
                                else
                                    tma_load_3d_pair(sb, &tm_c, fb, x, c * BT, it.h0 + pass - 1);
                                tma_load_2d_pair(sb + kTileAct, leader ? &tm_wg : &tm_wu, fb, x, j * BNEU);
                            } else {
                                if (pass == 0)
                                    tma_load_2d(sb, &tm_x, fb, x, c * BT);
                                else
                                    tma_load_3d(sb, &tm_c, fb, x, c * BT, it.h0 + pass - 1);
                                tma_load_2d(sb + kTileAct, &tm_wg, fb, x, j * BNEU);
                                tma_load_2d(sb + kTileAct + kTileW, &tm_wu, fb, x, j * BNEU);
                            }
                        };
                        const uint32_t fb = kPair ? full_lead + static_cast<uint32_t>(stage) * 8u
                                                  : smem_u32(&full_bar[stage]);
                        if constexpr (kBoxes == 1) {
                            // one k block per stage (the single form): the plain sequence
                            if (leader) mbar_arrive_expect_tx(smem_u32(&full_bar[stage]), (kPair ? 2u : 1u) * kStageBytes);
                            load_box(0, fb, ks * BK);
                        } else {
                            if (leader)
                                mbar_arrive_expect_tx(smem_u32(&full_bar[stage]),
                                                      (kPair ? 2u : 1u) * static_cast<uint32_t>(nb) * kBoxBytes);
                            if (nb == kBoxes) {
#pragma unroll
                                for (int hb = 0; hb < kBoxes; ++hb) load_box(hb, fb, (ks * kBoxes + hb) * BK);
                            } else {
                                for (int hb = 0; hb < nb; ++hb) load_box(hb, fb, (ks * kBoxes + hb) * BK);
                            }
                        }
                        if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                    }
                }
            }
        } else if (warp == 1 && lane == 0 && leader) {
            // -------------------------------------------------------------- MMA issuer (the even CTA of a pair)
            int stage = 0;
            uint32_t phase = 0;
            uint32_t pass_count = 0;   // over all units: selects the accumulator buffer
            bool ok = true;
            Item it;
            for (int i = 0; ok && get_item<kPair>(p, i, it); ++i) {
                const int passes = 1 + it.h1 - it.h0;
                for (int pass = 0; ok && pass < passes; ++pass, ++pass_count) {
                    const uint32_t buf = pass_count & 1u;
                    const uint32_t use = (pass_count >> 1) & 1u;
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
                        // the four 16-wide K steps of box hb; the first MMA of a pass overwrites
                        auto mma_box = [&](int hb, bool first) {
                            const uint64_t da = smem_desc_k128(st + hb * kBoxBytes);
                            // pair: W_gate here, W_up in the peer; single: W_gate then W_up, 256 rows
                            const uint64_t dw = smem_desc_k128(st + hb * kBoxBytes + kTileAct);
#pragma unroll
                            for (int kk = 0; kk < BK / UK; ++kk) {
                                // advance 16 elements = 32 bytes inside the swizzle atom
                                const uint64_t off = static_cast<uint64_t>((kk * UK * 2) >> 4);
                                const uint32_t accumulate = (first && kk == 0) ? 0u : 1u;
                                if constexpr (kPair)
                                    umma_bf16_pair(d_acc, da + off, dw + off, kIdesc, accumulate);
                                else
                                    umma_bf16(d_acc, da + off, dw + off, kIdesc, accumulate);
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
            }
            // Every MMA must have completed before TMEM or shared memory is released.
            if constexpr (kPair)
                umma_commit_pair(smem_u32(drain_bar), 3);
            else
                umma_commit(smem_u32(drain_bar));
        }
    } else {
        setmaxnreg_inc<kRegsLarge>();
        // ------------------------------------------------------------------ epilogue (every CTA)
        const int quad = warp & 3;                         // TMEM lanes 32*quad .. +31 = tokens
        const int half = (warp - kEpiWarp0) >> 2;          // neurons [64*half, 64*half + 64)
        const bool summer = (quad == 0);                   // adds the four quadrants of its half
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
        const uint32_t col_g = static_cast<uint32_t>(half * 64);          // gate columns of this half
        const uint32_t col_u = static_cast<uint32_t>(BNEU + half * 64);   // up columns of this half
        // The warp reads its 32 lanes (tokens) x 64 neurons as four chunks (h, cb): 16-lane half h,
        // 32-column block cb, one 16-lane load each of the gate and the up columns.  Register j =
        // 4 r + q of a chunk is (token 16 h + t/4 + 8 (q >> 1), neuron 32 cb + 8 r + 2 (t % 4) +
        // (q & 1)) for thread t, so a thread owns 4 tokens x 16 neurons; alpha and beta of its 64
        // pairs stay in registers for the whole unit, indexed [16 (2 h + cb) + j].
        float alpha[64], beta[64];
        uint32_t pass_count = 0, head_count = 0;
        bool ok = true;
        // sums over the thread's 4 tokens, per neuron: slot 8 cb + 2 r + (q & 1)
        auto acc_slot = [](int cb, int j) { return 8 * cb + 2 * (j >> 2) + (j & 1); };
        // Sums over the 8 lanes that share a thread's neurons (lanes differing in bits 2-4), in a
        // fixed order: afterwards v[0], v[1] hold neurons n(t), n(t) + 1 of the warp's 64,
        // n(t) = 32 ((t >> 4) & 1) + 8 ((t >> 2) & 3) + 2 (t & 3).
        auto butterfly8 = [&](float (&v)[16]) {
#pragma unroll
            for (int rd = 0; rd < 3; ++rd) {
                const int o = 16 >> rd;
                const int m = 8 >> rd;
                const bool upper = (lane & o) != 0;
#pragma unroll
                for (int i = 0; i < m; ++i) {
                    const float send = upper ? v[i] : v[i + m];
                    const float keep = upper ? v[i + m] : v[i];
                    v[i] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, o);
                }
            }
        };
        const int n_t = 32 * ((lane >> 4) & 1) + 8 * ((lane >> 2) & 3) + 2 * (lane & 3);
        // Adds this warp's 32-token sums (neurons n(t), n(t) + 1 in each thread) into the
        // four-quadrant sum of its half and, for the summing warps, writes the 64 results to dst.
        // Two shared-memory slots are used alternately; a slot is rewritten only after both
        // summing warps have read it.
        auto reduce_store = [&](float s0, float s1, float* dst) -> bool {
            const uint32_t slot = head_count & 1u;
            const uint32_t use = head_count >> 1;
            ++head_count;
            float* rs = red + slot * 4 * BNEU;
            if (!mbar_wait(smem_u32(&red_empty[slot]), (use & 1u) ^ 1u, abort_flag)) return false;
            *reinterpret_cast<float2*>(rs + quad * BNEU + half * 64 + n_t) = make_float2(s0, s1);
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&red_full[slot]));
            if (summer) {
                // the four quadrants of this half, in a fixed order
                if (!mbar_wait(smem_u32(&red_full[slot]), use & 1u, abort_flag)) return false;
#pragma unroll
                for (int b = 0; b < 2; ++b) {
                    const int n = half * 64 + 32 * b + lane;
                    dst[32 * b + lane] = ((rs[n] + rs[BNEU + n]) + rs[2 * BNEU + n]) + rs[3 * BNEU + n];
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&red_empty[slot]));
            }
            return true;
        };
        // Once the pass's last TMEM load has landed in registers the accumulator buffer is free:
        // release it (in the pair form an arrival on the even CTA's acc_empty) before the math
        // and the reduction.
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
        Item it;
        for (int i = 0; ok && get_item<kPair>(p, i, it); ++i) {
            int ucu, uj;
            unit_coords(p, it.unit, ucu, uj);
            // chunk uc = TC (the empty half of a last pair) has a slot of its own that the
            // reduce never reads
            const int uc = kPair ? 2 * ucu + static_cast<int>(rank) : ucu;
            const int64_t slot_unit = static_cast<int64_t>(uc) * p.NT + uj;   // partial slot: (chunk, tile)
            float* out = p.partial + (slot_unit * p.G + it.h0) * static_cast<int64_t>(BNEU);
            const int passes = 1 + it.h1 - it.h0;
            for (int pass = 0; pass < passes; ++pass, ++pass_count) {
                const uint32_t buf = pass_count & 1u;
                const uint32_t use = (pass_count >> 1) & 1u;
                if (!mbar_wait(smem_u32(&acc_full[buf]), use, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t acc = lane_base + buf * kBufCols;
                float sums[16];
#pragma unroll
                for (int k = 0; k < 16; ++k) sums[k] = 0.0f;
                if (pass == 0) {
                    // operating point; optionally the down-edge activation sums
                    const bool want_act = p.rms != nullptr && it.h0 == 0;
                    float ir2[4] = {0.0f, 0.0f, 0.0f, 0.0f};   // tokens 16 h + t/4 + 8 s, slot 2 h + s
                    if (want_act) {
#pragma unroll
                        for (int ts = 0; ts < 4; ++ts) {
                            const int64_t tok = static_cast<int64_t>(uc) * BT + quad * 32 + 16 * (ts >> 1) +
                                                (lane >> 2) + 8 * (ts & 1);
                            if (tok < p.T) {
                                const float r = p.rms[tok];
                                ir2[ts] = 1.0f / (r * r);
                            }
                        }
                    }
#pragma unroll
                    for (int ch = 0; ch < 4; ++ch) {
                        const int h = ch >> 1, cb = ch & 1;
                        float vg[16], vu[16];
                        const uint32_t lanes = static_cast<uint32_t>(16 * h) << 16;
                        tmem_ld_16x256b_x4(acc + lanes + col_g + 32u * cb, vg);
                        tmem_ld_16x256b_x4(acc + lanes + col_u + 32u * cb, vu);
                        tmem_wait_ld();
                        if (ch == 3) release(buf);
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            swiglu_alpha_beta(vg[j], vu[j], alpha[16 * ch + j], beta[16 * ch + j]);
                            const float act = beta[16 * ch + j] * vu[j];   // silu(g) u
                            sums[acc_slot(cb, j)] = fmaf(act * act, ir2[2 * h + ((j >> 1) & 1)], sums[acc_slot(cb, j)]);
                        }
                    }
                    if (!want_act) continue;
                    butterfly8(sums);
                    if (!reduce_store(sums[0], sums[1], p.partial_act + slot_unit * BNEU + half * 64)) { ok = false; break; }
                    continue;
                }
                // head pass: sums of Delta^2 over this warp's 32 tokens
#pragma unroll
                for (int ch = 0; ch < 4; ++ch) {
                    const int h = ch >> 1, cb = ch & 1;
                    float pg[16], pu[16];
                    const uint32_t lanes = static_cast<uint32_t>(16 * h) << 16;
                    tmem_ld_16x256b_x4(acc + lanes + col_g + 32u * cb, pg);
                    tmem_ld_16x256b_x4(acc + lanes + col_u + 32u * cb, pu);
                    tmem_wait_ld();
                    if (ch == 3) release(buf);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float dlt = fmaf(alpha[16 * ch + j], pg[j], beta[16 * ch + j] * pu[j]);
                        sums[acc_slot(cb, j)] = fmaf(dlt, dlt, sums[acc_slot(cb, j)]);
                    }
                }
                butterfly8(sums);
                if (!reduce_store(sums[0], sums[1], out + (pass - 1) * BNEU + half * 64)) { ok = false; break; }
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

// A[g,k] += sum over the heads h of row g (h = g*qpg ... g*qpg + qpg - 1) and
// over token chunks of the unit partials; qpg = 1 gives one row per head, qpg
// > 1 sums the query heads of a KV group (Sec. 3, per-query-head scores).
// Eight threads share one output: thread s sums the chunks c = s, s+8, ...
// (head by head), then the eight sums are added in a fixed order, so the
// result does not depend on scheduling.
constexpr int kReduceSplit = 8;
__global__ void affinity_reduce_kernel(const float* __restrict__ partial, float* __restrict__ A, int G, int N,
                                       int NT, int TC, const float* __restrict__ partial_act,
                                       float* __restrict__ act2, int qpg, int overwrite) {
    const int64_t total_a = static_cast<int64_t>(G / qpg) * N;
    const int64_t total = total_a + (act2 ? N : 0);
    const int s = threadIdx.x % kReduceSplit;
    const int64_t per_block = blockDim.x / kReduceSplit;
    for (int64_t base = blockIdx.x * per_block; base < total; base += static_cast<int64_t>(gridDim.x) * per_block) {
        const int64_t idx = base + threadIdx.x / kReduceSplit;
        float sum = 0.0f;
        if (idx < total_a) {
            const int g = static_cast<int>(idx / N);
            const int k = static_cast<int>(idx % N);
            const int j = k / BNEU, r = k % BNEU;
            for (int h = g * qpg; h < (g + 1) * qpg; ++h)
                for (int c = s; c < TC; c += kReduceSplit)
                    sum += partial[((static_cast<int64_t>(c) * NT + j) * G + h) * BNEU + r];
        } else if (idx < total) {
            const int k = static_cast<int>(idx - total_a);
            const int j = k / BNEU, r = k % BNEU;
            for (int c = s; c < TC; c += kReduceSplit) sum += partial_act[(static_cast<int64_t>(c) * NT + j) * BNEU + r];
        }
        // fixed-order tree over the 8 lanes of this output (lanes s^4, s^2, s^1)
        sum += __shfl_xor_sync(0xFFFFFFFFu, sum, 4);
        sum += __shfl_xor_sync(0xFFFFFFFFu, sum, 2);
        sum += __shfl_xor_sync(0xFFFFFFFFu, sum, 1);
        if (s == 0) {
            if (idx < total_a) A[idx] = overwrite ? sum : A[idx] + sum;
            else if (idx < total) act2[idx - total_a] = overwrite ? sum : act2[idx - total_a] + sum;
        }
    }
}

// The same sums with one thread per output, for a reduce confined to a few SMs: consecutive
// threads take consecutive neurons, so each token chunk's loads are coalesced.  The thread keeps
// the eight interleaved chunk sums c = s, s+8, ... (s = 0..7) that the eight threads of
// affinity_reduce_kernel form and adds them by the same tree (s^4, then s^2, then s^1), so the
// result is bitwise the same.
__global__ void affinity_reduce_rows_kernel(const float* __restrict__ partial, float* __restrict__ A, int G, int N,
                                            int NT, int TC, const float* __restrict__ partial_act,
                                            float* __restrict__ act2, int qpg, int overwrite) {
    const int64_t total_a = static_cast<int64_t>(G / qpg) * N;
    const int64_t total = total_a + (act2 ? N : 0);
    for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
         idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        float acc[kReduceSplit];
#pragma unroll
        for (int s = 0; s < kReduceSplit; ++s) acc[s] = 0.0f;
        if (idx < total_a) {
            const int g = static_cast<int>(idx / N);
            const int k = static_cast<int>(idx % N);
            const int j = k / BNEU, r = k % BNEU;
            for (int h = g * qpg; h < (g + 1) * qpg; ++h)
                for (int c0 = 0; c0 < TC; c0 += kReduceSplit) {
#pragma unroll
                    for (int s = 0; s < kReduceSplit; ++s)
                        if (c0 + s < TC)
                            acc[s] += partial[((static_cast<int64_t>(c0 + s) * NT + j) * G + h) * BNEU + r];
                }
        } else {
            const int k = static_cast<int>(idx - total_a);
            const int j = k / BNEU, r = k % BNEU;
            for (int c0 = 0; c0 < TC; c0 += kReduceSplit) {
#pragma unroll
                for (int s = 0; s < kReduceSplit; ++s)
                    if (c0 + s < TC) acc[s] += partial_act[(static_cast<int64_t>(c0 + s) * NT + j) * BNEU + r];
            }
        }
        // the tree of the shuffle reduction: lanes s and s^4, then s^2, then s^1
        const float sum = ((acc[0] + acc[4]) + (acc[2] + acc[6])) + ((acc[1] + acc[5]) + (acc[3] + acc[7]));
        if (idx < total_a) A[idx] = overwrite ? sum : A[idx] + sum;
        else act2[idx - total_a] = overwrite ? sum : act2[idx - total_a] + sum;
    }
}

// bf16 tensor map with a [box_rows x 64] box and 128-byte swizzle; out-of-range
// elements read as zero, which contributes nothing to any sum below.
static bool make_map(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims, const cuuint64_t* strides,
                     cuuint32_t box_rows) {
    auto enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint32_t box[3] = {static_cast<cuuint32_t>(BK), box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// partial slots: one per (token chunk, neuron tile), for an even number of chunks (the odd
// CTA of a last, half-empty pair stores into the extra chunk's slots)
static int64_t slot_units(int64_t T, int N) {
    const int64_t NT = (N + BNEU - 1) / BNEU;
    const int64_t TC = (T + BT - 1) / BT;
    return NT * ((TC + 1) / 2) * 2;
}

static size_t partial_bytes(int64_t T, int G, int N) {
    return static_cast<size_t>(slot_units(T, N)) * G * BNEU * sizeof(float);
}

// bytes of the header and the per-unit A partials (the down-edge activation
// partials, one more 128-float row per unit, come after them when requested)
size_t workspace_bytes(int64_t T, int d, int G, int N) {
    (void)d;
    return kWorkspaceHeader + partial_bytes(T, G, N);
}

size_t workspace_bytes_with_act(int64_t T, int d, int G, int N) {
    return align_up(workspace_bytes(T, d, G, N), 256) + static_cast<size_t>(slot_units(T, N)) * BNEU * sizeof(float);
}

// The fixed-order reduce of a workspace's unit partials into A (and act2 when the workspace
// holds the down-edge activation sums): G heads in the workspace, G / qpg rows of A.
// max_blocks > 0: that many blocks of 1024 threads (a reduce beside a kernel that holds every
// other SM); overwrite: store the sums instead of adding them.
int launch_reduce(const void* workspace, int64_t T, int d, int G, int N, float* A, float* act2, int qpg,
                  cudaStream_t stream, int max_blocks, int overwrite) {
    if (qpg < 1 || G % qpg) return DTP_ERR_ARG;
    const int NT = (N + BNEU - 1) / BNEU;
    const int TC = static_cast<int>((T + BT - 1) / BT);
    const float* partial = reinterpret_cast<const float*>(reinterpret_cast<const uint8_t*>(workspace) +
                                                          kWorkspaceHeader);
    const float* partial_act = act2 ? reinterpret_cast<const float*>(reinterpret_cast<const uint8_t*>(workspace) +
                                                                     align_up(workspace_bytes(T, d, G, N), 256))
                                    : nullptr;
    int dev = 0, sms = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const int64_t total = static_cast<int64_t>(G / qpg) * N + (act2 ? N : 0);
    if (max_blocks > 0) {
        const int64_t want = (total + 1023) / 1024;
        const int rblocks = static_cast<int>(want < max_blocks ? want : max_blocks);
        affinity_reduce_rows_kernel<<<rblocks, 1024, 0, stream>>>(partial, A, G, N, NT, TC, partial_act, act2, qpg,
                                                                  overwrite);
        DTP_CUDA_TRY(cudaGetLastError());
        return DTP_OK;
    }
    const int64_t outs_per_block = 256 / kReduceSplit;
    const int64_t want = (total + outs_per_block - 1) / outs_per_block;
    const int rblocks = static_cast<int>(want < 8 * sms ? want : 8 * sms);
    affinity_reduce_kernel<<<rblocks, 256, 0, stream>>>(partial, A, G, N, NT, TC, partial_act, act2, qpg, overwrite);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

// G heads of C; A receives G / qpg rows (qpg consecutive heads summed per row).  max_ctas > 0
// caps the persistent grid below one CTA per SM (leaving SMs to concurrent kernels); with
// defer_reduce the unit partials stay in the workspace for a later launch_reduce.
int launch_grouped(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N,
                   float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2, int qpg,
                   int max_ctas, int defer_reduce) {
    if (qpg < 1 || G % qpg) return DTP_ERR_ARG;
    CUtensorMap m_wg, m_wu, m_x, m_c;
    const cuuint64_t row_stride = static_cast<cuuint64_t>(d) * 2;
    cuuint64_t dw[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(N)};
    cuuint64_t dx[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T)};
    cuuint64_t dc[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(T), static_cast<cuuint64_t>(G)};
    cuuint64_t s2[1] = {row_stride};
    cuuint64_t s3[2] = {row_stride, row_stride * static_cast<cuuint64_t>(T)};
    if (!make_map(&m_wg, Wg, 2, dw, s2, BNEU) || !make_map(&m_wu, Wu, 2, dw, s2, BNEU) ||
        !make_map(&m_x, X, 2, dx, s2, BT) || !make_map(&m_c, C, 3, dc, s3, BT))
        return DTP_ERR_CUDA;

    Params p;
    p.G = G;
    p.NT = (N + BNEU - 1) / BNEU;
    p.TC = static_cast<int>((T + BT - 1) / BT);
    p.KB = (d + BK - 1) / BK;
    p.status = reinterpret_cast<int*>(workspace);
    p.partial = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(workspace) + kWorkspaceHeader);
    p.T = T;
    p.rms = (rms && act2) ? rms : nullptr;
    p.partial_act = p.rms ? reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(workspace) +
                                                     align_up(workspace_bytes(T, d, G, N), 256))
                          : nullptr;

    int dev = 0, sms = 0, l2 = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev));
    // CTA pairs when all weight tiles fit in half of L2 (no chunk grouping needed), single CTAs
    // otherwise (and wherever no cluster of two can be resident)
    const double tile_bytes = 2.0 * BNEU * d * 2.0;   // W_gate and W_up rows of one neuron tile
    const bool weights_fit = static_cast<double>(p.NT) * tile_bytes <= l2 / 2.0;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.stream = stream;
    cfg.attrs = attr;
    // CTA pairs resident at once, queried once per device (0: not yet; -1: none can be, for
    // instance on a partition too small for a cluster of two, and the single form runs instead)
    int resident = 0;
    if (weights_fit) {
        static std::atomic<int> resident_cache[64];
        resident = dev < 64 ? resident_cache[dev].load(std::memory_order_relaxed) : 0;
        if (resident == 0) {
            DTP_CUDA_TRY(cudaFuncSetAttribute(affinity_fo_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              static_cast<int>(Form<true>::kSmemBytes)));
            cfg.gridDim = dim3(static_cast<unsigned>(sms & ~1), 1, 1);
            cfg.dynamicSmemBytes = Form<true>::kSmemBytes;
            cfg.numAttrs = 1;
            if (cudaOccupancyMaxActiveClusters(&resident, affinity_fo_tc_kernel<true>, &cfg) != cudaSuccess ||
                resident < 1) {
                (void)cudaGetLastError();
                resident = -1;
            }
            if (dev < 64) resident_cache[dev].store(resident, std::memory_order_relaxed);
        }
    }
    const bool pair = resident > 0;
    auto kernel = pair ? affinity_fo_tc_kernel<true> : affinity_fo_tc_kernel<false>;
    const size_t smem = pair ? Form<true>::kSmemBytes : Form<false>::kSmemBytes;
    DTP_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
    attr[0].val.clusterDim.x = pair ? 2 : 1;
    cfg.dynamicSmemBytes = smem;
    cfg.numAttrs = pair ? 1 : 0;
    const int cap = (max_ctas > 0 && max_ctas < sms) ? max_ctas : sms;
    int workers;
    p.KS = pair ? (p.KB + Form<true>::kBoxes - 1) / Form<true>::kBoxes
                : (p.KB + Form<false>::kBoxes - 1) / Form<false>::kBoxes;
    if (pair) {
        p.TU = (p.TC + 1) / 2;
        // one CTA pair per two SMs (fewer under max_ctas, rounded down to pairs, at least one
        // pair), and no more pairs than can be resident at once
        workers = cap / 2 < resident ? cap / 2 : resident;
        if (workers < 1) workers = 1;
    } else {
        p.TU = p.TC;
        workers = cap;
    }
    p.units = static_cast<int64_t>(p.NT) * p.TU;
    if (p.units < workers) workers = static_cast<int>(p.units);
    // chunk grouping: keep the weight tiles of the units in flight within a third of L2
    p.cg = 1;
    if (!weights_fit)
        while (p.cg < 64 && p.cg < p.TU && (static_cast<double>(workers) / p.cg) * tile_bytes > l2 / 3.0) p.cg *= 2;
    p.full_rounds = static_cast<int>(p.units / workers);
    const int left = static_cast<int>(p.units - static_cast<int64_t>(p.full_rounds) * workers);
    p.split = left > 0 ? (workers / left < G ? workers / left : G) : 1;
    if (p.split < 1) p.split = 1;
    p.tail_items = left * p.split;
    cfg.gridDim = dim3(static_cast<unsigned>(pair ? 2 * workers : workers), 1, 1);
    DTP_CUDA_TRY(cudaLaunchKernelEx(&cfg, kernel, m_wg, m_wu, m_x, m_c, p));
    DTP_CUDA_TRY(cudaGetLastError());
    if (defer_reduce) return DTP_OK;
    return launch_reduce(workspace, T, d, G, N, A, p.rms ? act2 : nullptr, qpg, stream, 0, 0);
}

int launch(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A,
           void* workspace, cudaStream_t stream, const float* rms, float* act2) {
    return launch_grouped(X, C, Wg, Wu, T, d, G, N, A, workspace, stream, rms, act2, 1, 0, 0);
}

}  // namespace tc
}  // namespace dtp
