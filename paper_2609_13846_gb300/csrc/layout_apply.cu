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
//                        every row  (o columns, down columns)
// The gathers are pure data movement, bound by HBM: every byte is read once
// and written once with 16-byte accesses where the block width allows it.  A
// permutation entry outside [0, blocks) is not followed: the element is left
// unwritten and DTP_ERR_ARG is set in the status word.
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
