// layout_apply.cu -- applying a layout to the dense weights (Sec. 3): the
// optimiser's (h, nu) become permutations that list every device's KV groups
// and neurons contiguously, and the weights are gathered in that order so that
// device l's shard is the l-th contiguous slice.
//
//   layout_order_kernel  order[p] = the item at position p when the items are
//                        listed device by device, each device's in increasing
//                        index (one block per layer; a counting pass per
//                        device with a block-wide scan).
//   gather_rows_kernel   dst block b of rows = src block perm[b]  (q/k/v rows,
//                        gate/up rows)
//   gather_cols_kernel   dst column block b = src column block perm[b] in
//                        every row  (o columns; element-wise columns whose
//                        rows are not a multiple of 16 bytes)
//   gather_cols_staged_kernel  the same for element-wise columns (down
//                        columns, one per neuron) with 16-byte rows of up to
//                        32 KB: row tiles staged in shared memory, each
//                        thread's source offsets held in registers
// The gathers are pure data movement, bound by HBM: every byte is read once
// and written once with 16-byte accesses where the block width allows it.  A
// permutation entry outside [0, blocks) is not followed: the element is left
// unwritten (or, where elements are written as 16-byte words, set to zero) and
// DTP_ERR_ARG is set in the status word.
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace apply {

constexpr int kOrderThreads = 1024;

// One block per layer.  Labels outside [0, D) or a device holding other than
// n / D items (when `balanced`) set DTP_ERR_ARG in the status word.
__global__ void __launch_bounds__(kOrderThreads)
layout_order_kernel(const int32_t* __restrict__ labels, int n, int D, int balanced, int32_t* __restrict__ order,
                    int* status) {
    __shared__ int warp_tot[kOrderThreads / 32];
    __shared__ int base;
    const int32_t* lab = labels + static_cast<int64_t>(blockIdx.x) * n;
    int32_t* out = order + static_cast<int64_t>(blockIdx.x) * n;
    const int per = (n + kOrderThreads - 1) / kOrderThreads;
    const int k0 = threadIdx.x * per;
    const int k1 = min(n, k0 + per);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int bad = 0;
    for (int k = k0; k < k1; ++k)
        if (lab[k] < 0 || lab[k] >= D) bad = 1;
    bad = __syncthreads_or(bad);
    if (bad) {
        if (threadIdx.x == 0) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
        return;
    }
    if (threadIdx.x == 0) base = 0;
    __syncthreads();
    for (int l = 0; l < D; ++l) {
        int cnt = 0;
        for (int k = k0; k < k1; ++k) cnt += lab[k] == l;
        // exclusive scan of cnt over the block (thread order = item order)
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) warp_tot[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int w = warp_tot[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xFFFFFFFFu, w, o);
                if (lane >= o) w += y;
            }
            warp_tot[lane] = w;      // inclusive over warps
        }
        __syncthreads();
        int pos = base + (warp > 0 ? warp_tot[warp - 1] : 0) + incl - cnt;
        for (int k = k0; k < k1; ++k)
            if (lab[k] == l) out[pos++] = k;
        const int total = warp_tot[kOrderThreads / 32 - 1];
        __syncthreads();
        if (threadIdx.x == 0) {
            if (balanced && total != n / D) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
            base += total;
        }
        __syncthreads();
    }
}

// One warp per destination row (grid-stride over layers x rows); the lanes
// copy the row in V-sized pieces, so index arithmetic is per row, not per byte.

// dst[layer][b*B + r][:] = src[layer][perm[layer][b]*B + r][:], rows of row_bytes.
template <typename V>
__global__ void gather_rows_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst, int layers,
                                   int64_t rows, int64_t row_bytes, int block_rows, const int32_t* __restrict__ perm,
                                   int64_t perm_stride, int* status) {
    const int64_t nblocks = rows / block_rows;
    const int64_t vpr = row_bytes / static_cast<int64_t>(sizeof(V));
    const int64_t total_rows = rows * layers;
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    for (int64_t rr = blockIdx.x * static_cast<int64_t>(blockDim.x >> 5) + (threadIdx.x >> 5); rr < total_rows;
         rr += warps) {
        const int64_t layer = rr / rows;
        const int64_t row = rr - layer * rows;
        const int64_t b = row / block_rows;
        const int64_t pb = perm[layer * perm_stride + b];
        if (pb < 0 || pb >= nblocks) {
            if (lane == 0) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
            continue;
        }
        const int64_t srow = layer * rows + pb * block_rows + (row - b * block_rows);
        const V* s = reinterpret_cast<const V*>(src + srow * row_bytes);
        V* d = reinterpret_cast<V*>(dst + rr * row_bytes);
        for (int64_t v = lane; v < vpr; v += 32) d[v] = s[v];
    }
}

// dst[layer][r][b*B + c] = src[layer][r][perm[layer][b]*B + c].
//   kDirect: column blocks span whole 16-byte words, copied as uint4.
//   kPack:   elements E gathered one by one and written as 16-byte words.
//   kPlain:  elements E gathered and written one by one (rows not a multiple of 16 bytes).
enum ColMode { kDirect = 0, kPack = 1, kPlain = 2 };

template <typename E, int MODE>
__global__ void gather_cols_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst, int layers,
                                   int64_t rows, int64_t row_bytes, int64_t block_bytes,
                                   const int32_t* __restrict__ perm, int64_t perm_stride, int* status) {
    constexpr int64_t es = static_cast<int64_t>(sizeof(E));
    const int64_t nblocks = row_bytes / block_bytes;
    const int64_t block_elems = block_bytes / es;
    const int64_t total_rows = rows * layers;
    const int lane = threadIdx.x & 31;
    const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    for (int64_t rr = blockIdx.x * static_cast<int64_t>(blockDim.x >> 5) + (threadIdx.x >> 5); rr < total_rows;
         rr += warps) {
        const int64_t layer = rr / rows;
        const int32_t* pl = perm + layer * perm_stride;
        const uint8_t* s = src + rr * row_bytes;
        uint8_t* d = dst + rr * row_bytes;
        int bad = 0;
        if constexpr (MODE == kDirect) {
            const uint32_t bb = static_cast<uint32_t>(block_bytes);
            for (int64_t o = lane; o < row_bytes / 16; o += 32) {
                const uint32_t byte = static_cast<uint32_t>(o * 16);
                const uint32_t b = byte / bb;
                const int64_t pb = pl[b];
                if (pb < 0 || pb >= nblocks) { bad = 1; continue; }
                *reinterpret_cast<uint4*>(d + byte) =
                    *reinterpret_cast<const uint4*>(s + pb * block_bytes + (byte - b * bb));
            }
        } else if constexpr (MODE == kPack) {
            constexpr int kPer = static_cast<int>(16 / sizeof(E));
            const uint32_t be = static_cast<uint32_t>(block_elems);
            // one column per block and 16-byte aligned permutation rows: the kPer entries behind
            // an output word are read as whole 16-byte words (4 entries each)
            const bool vec_perm = kPer % 4 == 0 && block_elems == 1 &&
                                  (reinterpret_cast<uintptr_t>(pl) & 15) == 0;
            if (vec_perm) {
                for (int64_t o = lane; o < row_bytes / 16; o += 32) {
                    union { uint4 v; E e[kPer]; } w;
                    const int4* pv = reinterpret_cast<const int4*>(pl + o * kPer);
#pragma unroll
                    for (int q = 0; q < kPer / 4; ++q) {
                        const int4 p4 = pv[q];
                        const int32_t pe[4] = {p4.x, p4.y, p4.z, p4.w};
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const int64_t pb = pe[t];
                            if (pb < 0 || pb >= nblocks) { bad = 1; w.e[4 * q + t] = E(0); continue; }
                            w.e[4 * q + t] = reinterpret_cast<const E*>(s)[pb];
                        }
                    }
                    *reinterpret_cast<uint4*>(d + o * 16) = w.v;
                }
                if (bad) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
                continue;
            }
            for (int64_t o = lane; o < row_bytes / 16; o += 32) {
                union { uint4 v; E e[kPer]; } w;
#pragma unroll
                for (int i = 0; i < kPer; ++i) {
                    const uint32_t c = static_cast<uint32_t>(o * kPer + i);
                    const uint32_t b = c / be;
                    const int64_t pb = pl[b];
                    if (pb < 0 || pb >= nblocks) { bad = 1; w.e[i] = E(0); continue; }
                    w.e[i] = reinterpret_cast<const E*>(s)[pb * block_elems + (c - b * be)];
                }
                *reinterpret_cast<uint4*>(d + o * 16) = w.v;
            }
        } else {
            for (int64_t c = lane; c < row_bytes / es; c += 32) {
                const int64_t b = c / block_elems;
                const int64_t pb = pl[b];
                if (pb < 0 || pb >= nblocks) { bad = 1; continue; }
                reinterpret_cast<E*>(d)[c] = reinterpret_cast<const E*>(s)[pb * block_elems + (c - b * block_elems)];
            }
        }
        if (bad) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
    }
}

// Element-wise column gather staged through shared memory (rows of a multiple
// of 16 bytes, at most 32 KB, whose column blocks are not whole 16-byte words,
// e.g. one down_proj column per neuron).  Gathering such elements straight from
// global memory costs one 32-byte L1 sector per element; here each CTA
//   - streams tiles of R consecutive rows (contiguous in memory) into two
//     shared buffers with 1-D bulk copies (cp.async.bulk, completion counted on
//     an mbarrier), one thread issuing them,
//   - lets each thread own fixed 16-byte output words (ow = tid + w * 256,
//     w < WPT): when its range of tiles enters a layer, the thread reads the
//     permutation entries behind its words once and keeps their source offsets
//     in a staged row in registers (16 bits each, two per register),
//   - then, for every tile, walks the tile's rows gathering its words' elements
//     from shared memory and storing each word with one 16-byte write,
//     coalesced across the warp.
// CTAs take contiguous ranges of the layers x row-tiles list, so a thread reads
// the permutation again only when its range crosses into the next layer.
constexpr int kStagedThreads = 256;
constexpr int kStagedStages = 2;
constexpr int64_t kStagedTileTarget = 16 * 1024;   // bytes per staged row tile (at least one row)
constexpr int kStagedMaxWpt = 8;                    // rows of up to 8 * 256 words = 32 KB
constexpr uint32_t kNoOffset = 0xFFFFu;             // an entry that is not followed (rows < 64 KB)

struct StagedGeom {
    int64_t rows, row_bytes, block_elems, nblocks, perm_stride;
    int layers, tile_rows, tiles_per_layer;
    int64_t total_tiles;
};

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
        : "memory");
}

template <typename E, int WPT>
__global__ void __launch_bounds__(kStagedThreads)
gather_cols_staged_kernel(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst, StagedGeom g,
                          const int32_t* __restrict__ perm, int* status) {
    constexpr int kPer = static_cast<int>(16 / sizeof(E));   // elements per 16-byte word
    constexpr int kPairs = kPer / 2;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t bars[kStagedStages];
    __shared__ int abort_flag;
    const uint32_t row_bytes = static_cast<uint32_t>(g.row_bytes);
    const uint32_t stage_bytes = static_cast<uint32_t>(g.tile_rows) * row_bytes;
    const int tid = threadIdx.x;
    // this CTA's contiguous range of (layer, row tile) items
    const int64_t t_begin = g.total_tiles * blockIdx.x / gridDim.x;
    const int64_t t_end = g.total_tiles * (blockIdx.x + 1) / gridDim.x;
    if (t_begin >= t_end) return;
    if (tid == 0) {
        abort_flag = 0;
        for (int i = 0; i < kStagedStages; ++i) mbar_init(smem_u32(&bars[i]), 1);
        fence_mbar_init();
    }
    __syncthreads();

    auto tile_rows_of = [&](int64_t t) -> int {
        const int64_t r0 = (t % g.tiles_per_layer) * g.tile_rows;
        return static_cast<int>(min(static_cast<int64_t>(g.tile_rows), g.rows - r0));
    };
    auto issue = [&](int64_t t) {      // tile t into stage (t - t_begin) % S
        const int64_t layer = t / g.tiles_per_layer;
        const int64_t r0 = (t % g.tiles_per_layer) * g.tile_rows;
        const uint32_t bytes = static_cast<uint32_t>(tile_rows_of(t)) * row_bytes;
        const int st = static_cast<int>((t - t_begin) % kStagedStages);
        const uint32_t bar = smem_u32(&bars[st]);
        mbar_arrive_expect_tx(bar, bytes);
        bulk_g2s(smem_u32(smem + st * stage_bytes), src + (layer * g.rows + r0) * g.row_bytes, bytes, bar);
    };
    if (tid == 0)
        for (int64_t t = t_begin; t < t_end && t < t_begin + kStagedStages; ++t) issue(t);

    const int words = static_cast<int>(g.row_bytes / 16);
    const uint32_t be = static_cast<uint32_t>(g.block_elems);
    const uint32_t nblocks = static_cast<uint32_t>(g.nblocks);
    uint32_t off[WPT][kPairs];   // source byte offsets of this thread's words, two per register
    int64_t cur_layer = -1;
    int bad = 0;
    int64_t t = t_begin;
    for (; t < t_end; ++t) {
        const int64_t layer = t / g.tiles_per_layer;
        if (layer != cur_layer) {
            const int32_t* pl = perm + layer * g.perm_stride;
#pragma unroll
            for (int w = 0; w < WPT; ++w) {
                const int ow = tid + w * kStagedThreads;
#pragma unroll
                for (int i = 0; i < kPairs; ++i) {
                    uint32_t two[2] = {kNoOffset, kNoOffset};
                    if (ow < words) {
#pragma unroll
                        for (int k = 0; k < 2; ++k) {
                            const uint32_t c = static_cast<uint32_t>(ow) * kPer + 2 * i + k;
                            const uint32_t b = c / be;
                            const int32_t pb = __ldg(pl + b);
                            const bool ok = static_cast<uint32_t>(pb) < nblocks;
                            bad |= !ok;
                            if (ok) two[k] = (static_cast<uint32_t>(pb) * be + (c - b * be)) * sizeof(E);
                        }
                    }
                    off[w][i] = two[0] | (two[1] << 16);
                }
            }
            cur_layer = layer;
        }
        const int st = static_cast<int>((t - t_begin) % kStagedStages);
        const uint32_t parity = static_cast<uint32_t>(((t - t_begin) / kStagedStages) & 1);
        // the block leaves together: a wait that gave up makes every thread's wait give up
        // (shared abort flag), and the vote keeps the barrier counts of all threads equal
        const bool landed = mbar_wait(smem_u32(&bars[st]), parity, &abort_flag);
        if (!__syncthreads_and(landed)) break;
        const uint8_t* tile = smem + st * stage_bytes;
        const int nr = tile_rows_of(t);
        const int64_t r0 = (t % g.tiles_per_layer) * g.tile_rows;
        uint8_t* out = dst + (layer * g.rows + r0) * g.row_bytes;
#pragma unroll
        for (int w = 0; w < WPT; ++w) {
            const int ow = tid + w * kStagedThreads;
            if (ow >= words) continue;
            const uint8_t* rowp = tile;
            uint8_t* op = out + static_cast<int64_t>(ow) * 16;
            for (int r = 0; r < nr; ++r) {
                union { uint4 v; E e[kPer]; } wd;
#pragma unroll
                for (int i = 0; i < kPer; ++i) {
                    const uint32_t o = (i & 1) ? (off[w][i >> 1] >> 16) : (off[w][i >> 1] & 0xFFFFu);
                    wd.e[i] = o != kNoOffset ? *reinterpret_cast<const E*>(rowp + o) : E(0);
                }
                *reinterpret_cast<uint4*>(op) = wd.v;
                rowp += row_bytes;
                op += g.row_bytes;
            }
        }
        // every thread is done with this stage: refill it
        __syncthreads();
        if (tid == 0 && t + kStagedStages < t_end) issue(t + kStagedStages);
    }
    if (bad) atomicMin(status, static_cast<int>(DTP_ERR_ARG));
    if (t < t_end) {
        // a wait gave up: report it, then let the copies still in flight land before exiting
        __syncthreads();
        if (tid == 0) {
            atomicMin(status, static_cast<int>(DTP_ERR_NOT_CONVERGED));
            int ok = 1;
            for (int64_t u = t; u < t_end && u < t + kStagedStages && ok; ++u) {
                volatile int own = 0;
                const int su = static_cast<int>((u - t_begin) % kStagedStages);
                ok = mbar_wait(smem_u32(&bars[su]), static_cast<uint32_t>(((u - t_begin) / kStagedStages) & 1), &own);
            }
        }
        __syncthreads();
    }
}

static int grid_for(int64_t work) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                   cudaSuccess)
        return -1;
    const int64_t want = (work + 255) / 256;
    const int64_t cap = static_cast<int64_t>(sms) * 8;   // 8 resident 256-thread blocks per SM
    return static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
}

int launch_order(const int32_t* labels, int layers, int n, int D, int balanced, int32_t* order, void* workspace,
                 cudaStream_t stream) {
    layout_order_kernel<<<layers, kOrderThreads, 0, stream>>>(labels, n, D, balanced, order,
                                                             reinterpret_cast<int*>(workspace));
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

static int grid_for_rows(int64_t rows) {
    // 8 warps per block; at most 8 blocks per SM resident
    return grid_for(rows * 32);
}

int launch_rows(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int block_rows,
                const int32_t* perm, int64_t perm_stride, void* workspace, cudaStream_t stream) {
    int* status = reinterpret_cast<int*>(workspace);
    const bool wide = (row_bytes % 16) == 0 && (reinterpret_cast<uintptr_t>(src) & 15) == 0 &&
                      (reinterpret_cast<uintptr_t>(dst) & 15) == 0;
    const int grid = grid_for_rows(static_cast<int64_t>(layers) * rows);
    if (grid < 0) return DTP_ERR_CUDA;
    const auto* s = static_cast<const uint8_t*>(src);
    auto* d = static_cast<uint8_t*>(dst);
    if (wide)
        gather_rows_kernel<uint4><<<grid, 256, 0, stream>>>(s, d, layers, rows, row_bytes, block_rows, perm,
                                                            perm_stride, status);
    else
        gather_rows_kernel<uint8_t><<<grid, 256, 0, stream>>>(s, d, layers, rows, row_bytes, block_rows, perm,
                                                              perm_stride, status);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

template <typename E>
static void cols_by_elem(const uint8_t* s, uint8_t* d, int layers, int64_t rows, int64_t row_bytes,
                         int64_t block_bytes, const int32_t* perm, int64_t perm_stride, int* status, int grid,
                         bool pack, cudaStream_t stream) {
    if (pack)
        gather_cols_kernel<E, kPack><<<grid, 256, 0, stream>>>(s, d, layers, rows, row_bytes, block_bytes, perm,
                                                               perm_stride, status);
    else
        gather_cols_kernel<E, kPlain><<<grid, 256, 0, stream>>>(s, d, layers, rows, row_bytes, block_bytes, perm,
                                                                perm_stride, status);
}

// Element-wise path straight from global memory, for any element width.
static void cols_by_elem_any(const uint8_t* s, uint8_t* d, int layers, int64_t rows, int64_t row_bytes,
                             int64_t block_bytes, int elem_bytes, const int32_t* perm, int64_t perm_stride,
                             int* status, int grid, bool pack, cudaStream_t stream) {
    if (elem_bytes == 2)
        cols_by_elem<uint16_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, pack, stream);
    else if (elem_bytes == 4)
        cols_by_elem<uint32_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, pack, stream);
    else if (elem_bytes == 8)
        cols_by_elem<uint64_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, pack, stream);
    else
        cols_by_elem<uint8_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, pack, stream);
}

template <typename E, int WPT>
static int launch_staged_as(const uint8_t* s, uint8_t* d, const StagedGeom& g, size_t smem, const int32_t* perm,
                            int* status, cudaStream_t stream) {
    auto* fn = gather_cols_staged_kernel<E, WPT>;
    DTP_CUDA_TRY(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)));
    int dev = 0, sms = 0, per_sm = 0;
    DTP_CUDA_TRY(cudaGetDevice(&dev));
    DTP_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    DTP_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kStagedThreads, smem));
    if (per_sm < 1) return DTP_ERR_UNSUPPORTED;
    const int64_t cap = static_cast<int64_t>(sms) * per_sm;
    const int grid = static_cast<int>(g.total_tiles < cap ? g.total_tiles : cap);
    fn<<<grid, kStagedThreads, smem, stream>>>(s, d, g, perm, status);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

template <typename E>
static int launch_staged_words(const uint8_t* s, uint8_t* d, const StagedGeom& g, size_t smem, const int32_t* perm,
                               int* status, cudaStream_t stream) {
    const int64_t wpt = (g.row_bytes / 16 + kStagedThreads - 1) / kStagedThreads;
    if (wpt <= 1) return launch_staged_as<E, 1>(s, d, g, smem, perm, status, stream);
    if (wpt <= 2) return launch_staged_as<E, 2>(s, d, g, smem, perm, status, stream);
    if (wpt <= 4) return launch_staged_as<E, 4>(s, d, g, smem, perm, status, stream);
    return launch_staged_as<E, kStagedMaxWpt>(s, d, g, smem, perm, status, stream);
}

// Returns DTP_ERR_UNSUPPORTED (nothing launched) when the rows are wider than the staged kernel
// handles (32 KB); the caller then gathers from global memory.
static int launch_cols_staged(const uint8_t* s, uint8_t* d, int layers, int64_t rows, int64_t row_bytes,
                              int64_t block_elems, int elem_bytes, const int32_t* perm, int64_t perm_stride,
                              int* status, cudaStream_t stream) {
    if (row_bytes > static_cast<int64_t>(kStagedMaxWpt) * kStagedThreads * 16) return DTP_ERR_UNSUPPORTED;
    StagedGeom g;
    g.rows = rows;
    g.row_bytes = row_bytes;
    g.block_elems = block_elems;
    g.nblocks = row_bytes / elem_bytes / block_elems;
    g.perm_stride = perm_stride;
    g.layers = layers;
    int64_t tr = kStagedTileTarget / row_bytes;
    if (tr < 1) tr = 1;
    if (tr > rows) tr = rows;
    g.tile_rows = static_cast<int>(tr);
    g.tiles_per_layer = static_cast<int>((rows + tr - 1) / tr);
    g.total_tiles = static_cast<int64_t>(layers) * g.tiles_per_layer;
    const size_t smem = static_cast<size_t>(kStagedStages) * static_cast<size_t>(tr * row_bytes);
    if (g.total_tiles < 1) return DTP_ERR_UNSUPPORTED;
    switch (elem_bytes) {
        case 1: return launch_staged_words<uint8_t>(s, d, g, smem, perm, status, stream);
        case 2: return launch_staged_words<uint16_t>(s, d, g, smem, perm, status, stream);
        case 4: return launch_staged_words<uint32_t>(s, d, g, smem, perm, status, stream);
        default: return launch_staged_words<uint64_t>(s, d, g, smem, perm, status, stream);
    }
}

int launch_cols(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int64_t block_bytes,
                int elem_bytes, const int32_t* perm, int64_t perm_stride, void* workspace, cudaStream_t stream) {
    int* status = reinterpret_cast<int*>(workspace);
    const auto* s = static_cast<const uint8_t*>(src);
    auto* d = static_cast<uint8_t*>(dst);
    const int grid = grid_for_rows(static_cast<int64_t>(layers) * rows);
    if (grid < 0) return DTP_ERR_CUDA;
    const uintptr_t mis = (reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst));
    const bool rows16 = row_bytes % 16 == 0 && (mis & 15) == 0;
    if (rows16 && block_bytes % 16 == 0) {
        gather_cols_kernel<uint4, kDirect><<<grid, 256, 0, stream>>>(s, d, layers, rows, row_bytes, block_bytes, perm,
                                                                     perm_stride, status);
    } else if (rows16 && (elem_bytes == 1 || elem_bytes == 2 || elem_bytes == 4 || elem_bytes == 8) &&
               (mis & (elem_bytes - 1)) == 0 && block_bytes % elem_bytes == 0) {
        const int st = launch_cols_staged(s, d, layers, rows, row_bytes, block_bytes / elem_bytes, elem_bytes, perm,
                                          perm_stride, status, stream);
        if (st != DTP_ERR_UNSUPPORTED) return st;
        cols_by_elem_any(s, d, layers, rows, row_bytes, block_bytes, elem_bytes, perm, perm_stride, status, grid,
                         rows16, stream);
    } else if (elem_bytes == 2 && (mis & 1) == 0) {
        cols_by_elem<uint16_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, rows16,
                               stream);
    } else if (elem_bytes == 4 && (mis & 3) == 0) {
        cols_by_elem<uint32_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, rows16,
                               stream);
    } else if (elem_bytes == 8 && (mis & 7) == 0) {
        cols_by_elem<uint64_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid, rows16,
                               stream);
    } else {
        cols_by_elem<uint8_t>(s, d, layers, rows, row_bytes, block_bytes, perm, perm_stride, status, grid,
                              rows16 && elem_bytes == 1, stream);
    }
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace apply
}  // namespace dtp
