// search.cu -- the layout optimiser of Sec. 3 ("Objective", "Optimiser") on
// the GPU: coordinate ascent over balanced head partitions h and balanced
// neuron assignments nu of one layer, maximising the co-located up-edge mass.
//
// One thread block (1024 threads) per layer; the layers of a batch are
// independent because the up-edge objective decouples across layers.
//
// Exactness.  A is mapped to q[g,k] = floor(A[g,k] * 2^(40-e)) (max A < 2^e),
// computed from the fp32 bit pattern with integer shifts, and every score is
// an int64 sum, so no summation order can change a decision.
//
// Neuron step (exact balanced linear assignment, lexicographically smallest
// optimum), gain M[k,l] = sum over heads g with h(g) == l of q[g,k]:
//   D == 2  device 0 takes the N/2 largest M[k,0]-M[k,1], lower index first on
//           ties: one block-wide radix selection of packed (difference, index)
//           keys.
//   D >  2  (a) device prices pi from Gauss-Seidel sweeps (until the excess
//           over N/D is at most 2D neurons, at most kMaxSweeps), each price set
//           by a radix selection so that about N/D neurons prefer its device;
//           (b) every neuron to its best device at those prices -- optimal for
//           the resulting device counts by complementary slackness;
//           (c) successive shortest paths on the D-node exchange graph
//           (w[a][b] = best gain of moving one neuron from a to b) move one
//           unit of excess per path until all counts equal N/D: each path is
//           a maximum-gain path, so optimality for the counts is kept and the
//           final assignment is optimal;
//           (d) canonicalisation: for k = 0, 1, ..., move k to the smallest
//           device l < nu(k) that a zero-gain exchange cycle through neurons
//           > k allows; the result is the lexicographically smallest optimum.
// Head step: B[g,l] = sum over neurons on l of q[g,k]; every labelled balanced
// partition (H!/((H/D)!)^D of them) is scored by a slice of the block and the
// best, lexicographically smallest on ties, is kept.
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace search {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int DMAX = 8;
constexpr int GMAX = 16;
constexpr int kFixedBits = 40;
constexpr int kIdxBits = 18;                       // N <= 2^18
constexpr int64_t kValBias = int64_t(1) << 45;     // |gain| < 2^44 (H_kv <= 16): fits the 46-bit field
constexpr int64_t kNegInf = INT64_MIN / 4;
constexpr int kMaxSweeps = 16;                      // price sweeps before the exact repair
constexpr size_t kSmemBudget = 220 * 1024;         // dynamic smem for M, nu and (if it fits) A

struct Shared {
    uint64_t w[DMAX][DMAX];        // exchange-graph keys (0 = no neuron on the source device)
    int64_t P[DMAX][DMAX];         // all-pairs max-gain paths
    int64_t B[GMAX * DMAX];        // head-step column sums
    int64_t pi[DMAX];              // device prices
    int count[DMAX];
    unsigned int hist[256];
    int64_t red_i64[kWarps];
    int red_int[kWarps];
    uint64_t sel_prefix;
    long long sel_rank;
    int64_t total, J, Jprev;
    int h[GMAX];
    int hn[GMAX];                  // next layer's head partition (whole-model search)
    int status;
    int flag;
    int kstar;
    int best_idx;
};

// ---------------------------------------------------------------- helpers --

__device__ __forceinline__ size_t align_up_dev(size_t x, size_t a) { return (x + a - 1) / a * a; }

// f(i, a[i]) for every i < n, the block's threads taking consecutive elements: 16-byte loads of
// four elements when a is 16-byte aligned (the tail, and unaligned arrays, element by element).
// Every caller's result is independent of the visiting order (a max, an exact integer sum, or an
// element-wise copy).
template <class F>
__device__ __forceinline__ void for_each_a(const float* __restrict__ a, int64_t n, F&& f) {
    int64_t head = 0;
    if ((reinterpret_cast<uintptr_t>(a) & 15u) == 0) {
        const int64_t n4 = n >> 2;
        const float4* a4 = reinterpret_cast<const float4*>(a);
        for (int64_t i = threadIdx.x; i < n4; i += kThreads) {
            const float4 v = a4[i];
            f(4 * i, v.x);
            f(4 * i + 1, v.y);
            f(4 * i + 2, v.z);
            f(4 * i + 3, v.w);
        }
        head = n4 << 2;
    }
    for (int64_t i = head + threadIdx.x; i < n; i += kThreads) f(i, a[i]);
}

// floor(a * 2^(bits-e)) for a finite a >= 0, by shifting the fp32 significand.
__device__ __forceinline__ int64_t quantize_bits(float a, int e, int bits) {
    const uint32_t b = __float_as_uint(a);
    const uint32_t ex = (b >> 23) & 0xFFu;
    uint64_t m = b & 0x7FFFFFu;
    int E;
    if (ex == 0) {
        E = -149;
    } else {
        m |= 0x800000u;
        E = static_cast<int>(ex) - 150;
    }
    const int s = E + bits - e;
    if (s >= 0) return static_cast<int64_t>(m << s);
    if (s <= -40) return 0;
    return static_cast<int64_t>(m >> (-s));
}

__device__ __forceinline__ int64_t quantize(float a, int e) { return quantize_bits(a, e, kFixedBits); }

__device__ __forceinline__ uint64_t pack_gain(int64_t v, int k) {
    return (static_cast<uint64_t>(v + kValBias) << kIdxBits) |
           static_cast<uint64_t>((1 << kIdxBits) - 1 - k);
}
__device__ __forceinline__ int64_t gain_of(uint64_t key) {
    return static_cast<int64_t>(key >> kIdxBits) - kValBias;
}
__device__ __forceinline__ int index_of(uint64_t key) {
    return (1 << kIdxBits) - 1 - static_cast<int>(key & ((1u << kIdxBits) - 1));
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t x) {
    const uint32_t hi = static_cast<uint32_t>(x >> 32);
    const uint32_t mhi = __reduce_max_sync(0xFFFFFFFFu, hi);
    const uint32_t lo = (hi == mhi) ? static_cast<uint32_t>(x) : 0u;
    const uint32_t mlo = __reduce_max_sync(0xFFFFFFFFu, lo);
    return (static_cast<uint64_t>(mhi) << 32) | mlo;
}

__device__ __forceinline__ int64_t warp_sum_i64(int64_t x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    return x;
}

__device__ int64_t block_sum_i64(int64_t x, Shared& sh) {
    x = warp_sum_i64(x);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) sh.red_i64[warp] = x;
    __syncthreads();
    int64_t t = 0;
    for (int i = 0; i < kWarps; ++i) t += sh.red_i64[i];
    return t;
}

__device__ int64_t block_max_i64(int64_t x, Shared& sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t y = __shfl_xor_sync(0xFFFFFFFFu, x, o);
        x = y > x ? y : x;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) sh.red_i64[warp] = x;
    __syncthreads();
    int64_t t = sh.red_i64[0];
    for (int i = 1; i < kWarps; ++i) t = sh.red_i64[i] > t ? sh.red_i64[i] : t;
    return t;
}

__device__ int block_min_int(int x, Shared& sh) {
    x = static_cast<int>(__reduce_min_sync(0xFFFFFFFFu, static_cast<unsigned>(x)));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) sh.red_int[warp] = x;
    __syncthreads();
    int t = sh.red_int[0];
    for (int i = 1; i < kWarps; ++i) t = sh.red_int[i] < t ? sh.red_int[i] : t;
    return t;
}

// The r-th largest (1-based) of the n keys key(0..n-1), by an 8-bit
// most-significant-digit radix selection.  Collective over the block.
template <class KeyFn>
__device__ uint64_t block_select_desc(int n, long long r, KeyFn key, Shared& sh) {
    uint64_t prefix = 0;
    if (threadIdx.x == 0) sh.sel_rank = r;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = threadIdx.x; i < 256; i += kThreads) sh.hist[i] = 0;
        __syncthreads();
        const uint64_t hi_mask = (shift == 56) ? 0ull : (~0ull << (shift + 8));
        for (int i = threadIdx.x; i < n; i += kThreads) {
            const uint64_t kv = key(i);
            const bool match = (kv & hi_mask) == (prefix & hi_mask);
            const unsigned bin = match ? static_cast<unsigned>((kv >> shift) & 255u) : 256u;
            const unsigned peers = __match_any_sync(__activemask(), bin);
            if (match && (__ffs(peers) - 1) == (threadIdx.x & 31)) atomicAdd(&sh.hist[bin], __popc(peers));
        }
        __syncthreads();
        if (threadIdx.x < 32) {
            // lane L owns bins [248 - 8L, 255 - 8L], scanned from the top
            const int lane = threadIdx.x;
            unsigned cnt = 0;
            for (int b = 0; b < 8; ++b) cnt += sh.hist[255 - 8 * lane - b];
            unsigned incl = cnt;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += y;
            }
            const long long rr = sh.sel_rank;
            const bool here = (incl >= rr) && (incl - cnt < rr);
            const unsigned who = __ballot_sync(0xFFFFFFFFu, here);
            if (here) {
                long long left = rr - static_cast<long long>(incl - cnt);
                for (int b = 0; b < 8; ++b) {
                    const int bin = 255 - 8 * lane - b;
                    if (left <= static_cast<long long>(sh.hist[bin])) {
                        sh.sel_prefix = prefix | (static_cast<uint64_t>(bin) << shift);
                        sh.sel_rank = left;
                        break;
                    }
                    left -= sh.hist[bin];
                }
            }
            if (who == 0u && lane == 0) sh.status = DTP_ERR_NOT_CONVERGED;  // rank out of range
        }
        __syncthreads();
        prefix = sh.sel_prefix;
        __syncthreads();
    }
    return prefix;
}

struct Layer {
    const float* A;   // the layer's affinities: a shared-memory copy when it fits, else global
    int G, N, D, cap, e;
    int64_t* M;   // [N][D]
    int32_t* nu;  // [N]
    uint64_t* keys = nullptr;   // [N] selection keys, when M lives in global memory (else null)
};

// Bytes of M [N][D] int64 and nu [N] int32 (256-aligned); a layer kept in global memory also
// has N uint64 selection keys after them.
__host__ __device__ inline size_t mnu_bytes(int N, int D) {
    const size_t b = static_cast<size_t>(N) * D * sizeof(int64_t) + static_cast<size_t>(N) * sizeof(int32_t);
    return (b + 255) / 256 * 256;
}
__host__ __device__ inline size_t global_layer_bytes(int N, int D) {
    return mnu_bytes(N, D) + (static_cast<size_t>(N) * sizeof(uint64_t) + 255) / 256 * 256;
}

template <int DT>
__device__ void build_gain(const Layer& L, Shared& sh) {
    for (int k = threadIdx.x; k < L.N; k += kThreads) {
        float a[GMAX];
#pragma unroll
        for (int g = 0; g < GMAX; ++g) a[g] = g < L.G ? L.A[static_cast<int64_t>(g) * L.N + k] : 0.0f;
        int64_t m[DT];
#pragma unroll
        for (int l = 0; l < DT; ++l) m[l] = 0;
#pragma unroll
        for (int g = 0; g < GMAX; ++g) {
            if (g >= L.G) break;
            const int64_t q = quantize(a[g], L.e);
            const int hg = sh.h[g];
#pragma unroll
            for (int l = 0; l < DT; ++l)
                if (l == hg) m[l] += q;
        }
#pragma unroll
        for (int l = 0; l < DT; ++l) L.M[static_cast<int64_t>(k) * DT + l] = m[l];
    }
    __syncthreads();
}

// Exchange graph over neurons with index > lo: sh.w[a][b] = packed
// (max gain of moving such a neuron from a to b, lowest index among ties).
template <int DT>
__device__ void exchange_graph(const Layer& L, Shared& sh, int lo) {
    if (threadIdx.x < DMAX * DMAX) sh.w[threadIdx.x / DMAX][threadIdx.x % DMAX] = 0;
    __syncthreads();
    for (int a = 0; a < DT; ++a) {
        uint64_t best[DT];
#pragma unroll
        for (int b = 0; b < DT; ++b) best[b] = 0;
        for (int k = threadIdx.x; k < L.N; k += kThreads) {
            if (k <= lo || L.nu[k] != a) continue;
            const int64_t* mk = L.M + static_cast<int64_t>(k) * DT;
            const int64_t ma = mk[a];
#pragma unroll
            for (int b = 0; b < DT; ++b)
                if (b != a) {
                    const uint64_t key = pack_gain(mk[b] - ma, k);
                    best[b] = key > best[b] ? key : best[b];
                }
        }
#pragma unroll
        for (int b = 0; b < DT; ++b)
            if (b != a) {
                const uint64_t r = warp_max_u64(best[b]);
                if ((threadIdx.x & 31) == 0 && r) atomicMax(reinterpret_cast<unsigned long long*>(&sh.w[a][b]), r);
            }
    }
    __syncthreads();
}

__device__ void count_devices(const Layer& L, Shared& sh) {
    if (threadIdx.x < DMAX) sh.count[threadIdx.x] = 0;
    __syncthreads();
    for (int k = threadIdx.x; k < L.N; k += kThreads) atomicAdd(&sh.count[L.nu[k]], 1);
    __syncthreads();
}

// Best device of neuron k at prices pi (lowest index on ties).
template <int DT>
__device__ __forceinline__ int best_device(const Layer& L, const Shared& sh, int k) {
    const int64_t* mk = L.M + static_cast<int64_t>(k) * DT;
    int best = 0;
    int64_t bv = mk[0] - sh.pi[0];
#pragma unroll
    for (int l = 1; l < DT; ++l) {
        const int64_t v = mk[l] - sh.pi[l];
        if (v > bv) bv = v, best = l;
    }
    return best;
}

// ------------------------------------------------------------ neuron steps --

__device__ void neuron_step_d2(const Layer& L, Shared& sh) {
    const int64_t* M = L.M;
    auto key = [M](int k) -> uint64_t { return pack_gain(M[2 * k] - M[2 * k + 1], k); };
    const uint64_t tau = block_select_desc(L.N, L.cap, key, sh);
    for (int k = threadIdx.x; k < L.N; k += kThreads) L.nu[k] = key(k) >= tau ? 0 : 1;
    __syncthreads();
}

// Thread 0: max-gain path by Bellman-Ford over the D devices, from the devices
// in `src` (dist 0) and relaxing the exchange graph sh.w.  Returns pred[].
__device__ void bellman_ford(const Layer& L, const Shared& sh, unsigned src, int64_t* dist, int* pred) {
    for (int a = 0; a < L.D; ++a) {
        dist[a] = (src >> a) & 1u ? 0 : kNegInf;
        pred[a] = -1;
    }
    for (int round = 0; round < L.D - 1; ++round)
        for (int a = 0; a < L.D; ++a) {
            if (dist[a] == kNegInf) continue;
            for (int b = 0; b < L.D; ++b) {
                if (b == a || sh.w[a][b] == 0) continue;
                const int64_t nd = dist[a] + gain_of(sh.w[a][b]);
                if (nd > dist[b]) dist[b] = nd, pred[b] = a;
            }
        }
}

// Thread 0: move the best neuron of each edge of the path ending at `end`.
__device__ bool apply_path(const Layer& L, const Shared& sh, const int* pred, int end) {
    int v = end, steps = 0;
    while (pred[v] >= 0) {
        if (++steps > L.D) return false;
        const int a = pred[v];
        L.nu[index_of(sh.w[a][v])] = v;
        v = a;
    }
    return true;
}

template <int DT>
__device__ void neuron_step_general(const Layer& L, Shared& sh) {
    const int N = L.N, D = L.D, cap = L.cap;
    // (a) price sweeps
    for (int sweep = 0; sweep < kMaxSweeps; ++sweep) {
        if (threadIdx.x < DMAX) sh.count[threadIdx.x] = 0;
        __syncthreads();
        for (int k = threadIdx.x; k < N; k += kThreads) atomicAdd(&sh.count[best_device<DT>(L, sh, k)], 1);
        __syncthreads();
        int excess = 0;
        for (int l = 0; l < D; ++l) excess += sh.count[l] > cap ? sh.count[l] - cap : 0;
        if (excess <= 2 * D) break;
        for (int l = 0; l < D; ++l) {
            const int64_t* M = L.M;
            const int64_t* pi = sh.pi;
            auto key = [M, pi, l, D](int k) -> uint64_t {
                const int64_t* mk = M + static_cast<int64_t>(k) * D;
                int64_t alt = kNegInf;
                for (int m = 0; m < D; ++m)
                    if (m != l) alt = (mk[m] - pi[m]) > alt ? (mk[m] - pi[m]) : alt;
                const int64_t v = mk[l] - alt;
                return static_cast<uint64_t>(v) ^ (1ull << 63);
            };
            uint64_t t;
            if (L.keys) {
                // M is in global memory: form every key once, then the selection's passes read one
                // word per neuron instead of D
                for (int k = threadIdx.x; k < N; k += kThreads) L.keys[k] = key(k);
                __syncthreads();
                const uint64_t* ks = L.keys;
                t = block_select_desc(N, cap + 1, [ks](int k) -> uint64_t { return ks[k]; }, sh);
            } else {
                t = block_select_desc(N, cap + 1, key, sh);
            }
            if (threadIdx.x == 0) sh.pi[l] = static_cast<int64_t>(t ^ (1ull << 63));
            __syncthreads();
        }
    }
    // (b) assignment at the current prices
    for (int k = threadIdx.x; k < N; k += kThreads) L.nu[k] = best_device<DT>(L, sh, k);
    __syncthreads();
    count_devices(L, sh);
    // (c) successive shortest paths until balanced
    for (int aug = 0; aug < 4 * N + 16; ++aug) {
        if (threadIdx.x == 0) {
            int ex = 0;
            for (int l = 0; l < D; ++l) ex += sh.count[l] > cap ? 1 : 0;
            sh.flag = ex;
        }
        __syncthreads();
        if (sh.flag == 0) break;
        exchange_graph<DT>(L, sh, -1);
        if (threadIdx.x == 0) {
            unsigned src = 0;
            for (int l = 0; l < D; ++l)
                if (sh.count[l] > cap) src |= 1u << l;
            int64_t dist[DMAX];
            int pred[DMAX];
            bellman_ford(L, sh, src, dist, pred);
            int e = -1;
            for (int l = 0; l < D; ++l)
                if (sh.count[l] < cap && dist[l] != kNegInf && (e < 0 || dist[l] > dist[e])) e = l;
            int s = e;
            for (int steps = 0; e >= 0 && pred[s] >= 0 && steps <= D; ++steps) s = pred[s];
            if (e < 0 || !apply_path(L, sh, pred, e)) {
                sh.status = DTP_ERR_NOT_CONVERGED;
            } else {
                sh.count[s] -= 1;
                sh.count[e] += 1;
            }
        }
        __syncthreads();
        if (sh.status != DTP_OK) return;
    }
    if (threadIdx.x == 0)
        for (int l = 0; l < D; ++l)
            if (sh.count[l] != cap) sh.status = DTP_ERR_NOT_CONVERGED;
    __syncthreads();
    if (sh.status != DTP_OK) return;

    // (d) lexicographically smallest optimum
    int kstart = 0;
    for (int round = 0; round < N + 1; ++round) {
        exchange_graph<DT>(L, sh, -1);
        if (threadIdx.x == 0) {
            for (int a = 0; a < D; ++a)
                for (int b = 0; b < D; ++b)
                    sh.P[a][b] = (a == b) ? 0 : (sh.w[a][b] ? gain_of(sh.w[a][b]) : kNegInf);
            for (int c = 0; c < D; ++c)
                for (int a = 0; a < D; ++a)
                    for (int b = 0; b < D; ++b)
                        if (sh.P[a][c] != kNegInf && sh.P[c][b] != kNegInf && sh.P[a][c] + sh.P[c][b] > sh.P[a][b])
                            sh.P[a][b] = sh.P[a][c] + sh.P[c][b];
            for (int a = 0; a < D; ++a)
                if (sh.P[a][a] > 0) sh.status = DTP_ERR_NOT_CONVERGED;  // a positive cycle: not optimal
            // prices for the next neuron step: longest paths from a zero root
            for (int a = 0; a < D; ++a) sh.pi[a] = 0;
            for (int a = 0; a < D; ++a)
                for (int b = 0; b < D; ++b)
                    if (sh.P[a][b] != kNegInf && sh.P[a][b] > sh.pi[b]) sh.pi[b] = sh.P[a][b];
        }
        __syncthreads();
        if (sh.status != DTP_OK) return;
        int cand = N;
        for (int k = kstart + static_cast<int>(threadIdx.x); k < N; k += kThreads) {
            const int t = L.nu[k];
            const int64_t* mk = L.M + static_cast<int64_t>(k) * D;
            for (int l = 0; l < t; ++l)
                if (sh.P[l][t] != kNegInf && mk[l] - mk[t] + sh.P[l][t] == 0) { cand = k; break; }
            if (cand < N) break;
        }
        const int kstar = block_min_int(cand, sh);
        if (kstar >= N) break;
        exchange_graph<DT>(L, sh, kstar);
        if (threadIdx.x == 0) {
            const int t = L.nu[kstar];
            const int64_t* mk = L.M + static_cast<int64_t>(kstar) * D;
            for (int l = 0; l < t; ++l) {
                int64_t dist[DMAX];
                int pred[DMAX];
                bellman_ford(L, sh, 1u << l, dist, pred);
                if (dist[t] != kNegInf && mk[l] - mk[t] + dist[t] == 0) {
                    if (!apply_path(L, sh, pred, t)) sh.status = DTP_ERR_NOT_CONVERGED;
                    L.nu[kstar] = l;
                    break;
                }
            }
        }
        __syncthreads();
        if (sh.status != DTP_OK) return;
        kstart = kstar + 1;
    }
}

// --------------------------------------------------------------- head step --

// The idx-th labelled balanced partition in lexicographic order of
// (h(0), h(1), ...).  With W the number of completions of the current prefix,
// choosing label l at a position with R groups left leaves W * cnt[l] / R
// completions (an exact multinomial); all counts stay below 2^30.
__device__ void unrank_partition(uint32_t idx, uint32_t n_parts, int G, int D, int* h) {
    int cnt[DMAX];
    for (int l = 0; l < D; ++l) cnt[l] = G / D;
    uint32_t W = n_parts;
    for (int g = 0; g < G; ++g) {
        const uint32_t R = static_cast<uint32_t>(G - g);
        for (int l = 0; l < D; ++l) {
            if (cnt[l] == 0) continue;
            const uint32_t w = W * static_cast<uint32_t>(cnt[l]) / R;
            if (idx < w) {
                h[g] = l;
                W = w;
                cnt[l] -= 1;
                break;
            }
            idx -= w;
        }
    }
}

__device__ bool next_partition(int* h, int G) {
    int i = G - 2;
    while (i >= 0 && h[i] >= h[i + 1]) --i;
    if (i < 0) return false;
    int j = G - 1;
    while (h[j] <= h[i]) --j;
    int t = h[i]; h[i] = h[j]; h[j] = t;
    for (int a = i + 1, b = G - 1; a < b; ++a, --b) t = h[a], h[a] = h[b], h[b] = t;
    return true;
}

// (score, index) with the larger score, then the smaller index.
__device__ __forceinline__ void better(int64_t& s, int& i, int64_t s2, int i2) {
    if (s2 > s || (s2 == s && i2 < i)) s = s2, i = i2;
}

// Head-step column sums of one layer: B[g,l] = sum over neurons k on device l of q[g,k].
template <int DT>
__device__ void head_sums(const Layer& L, Shared& sh) {
    const int G = L.G, D = L.D;
    if (threadIdx.x < GMAX * DMAX) sh.B[threadIdx.x] = 0;
    __syncthreads();
    // B[g,l]: whole warps per head, each thread a strided slice of the neurons
    const int warps_per_head = kWarps / G;                 // G <= 16, so >= 2
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = warp / warps_per_head;
    if (g < G) {
        const int tph = warps_per_head * 32;
        const int sub = (warp % warps_per_head) * 32 + lane;
        int64_t acc[DT];
#pragma unroll
        for (int l = 0; l < DT; ++l) acc[l] = 0;
        const float* a = L.A + static_cast<int64_t>(g) * L.N;
        for (int k = sub; k < L.N; k += tph) {
            const int64_t q = quantize(a[k], L.e);
            const int l0 = L.nu[k];
#pragma unroll
            for (int l = 0; l < DT; ++l)
                if (l == l0) acc[l] += q;
        }
#pragma unroll
        for (int l = 0; l < DT; ++l) {
            const int64_t v = warp_sum_i64(acc[l]);
            if (lane == 0 && v)
                atomicAdd(reinterpret_cast<unsigned long long*>(&sh.B[g * D + l]), static_cast<unsigned long long>(v));
        }
    }
    __syncthreads();
}

// The best labelled balanced partition for the column sums in sh.B: every
// partition scored by a slice of the block, each thread a contiguous range in
// lexicographic order; result (lexicographically smallest among ties) in
// sh.h, its score in sh.J.
__device__ void choose_partition(const Layer& L, Shared& sh, uint32_t n_parts) {
    const int G = L.G, D = L.D;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t lo = static_cast<uint32_t>((static_cast<uint64_t>(n_parts) * threadIdx.x) / kThreads);
    const uint32_t hi = static_cast<uint32_t>((static_cast<uint64_t>(n_parts) * (threadIdx.x + 1)) / kThreads);
    int64_t best = kNegInf;
    int best_idx = 0x7FFFFFFF;
    if (lo < hi) {
        int hh[GMAX];
        unrank_partition(lo, n_parts, G, D, hh);
        for (uint32_t idx = lo; idx < hi; ++idx) {
            int64_t s = 0;
            for (int gg = 0; gg < G; ++gg) s += sh.B[gg * D + hh[gg]];
            if (s > best) best = s, best_idx = static_cast<int>(idx);
            if (idx + 1 < hi) next_partition(hh, G);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t s2 = __shfl_xor_sync(0xFFFFFFFFu, best, o);
        const int i2 = __shfl_xor_sync(0xFFFFFFFFu, best_idx, o);
        better(best, best_idx, s2, i2);
    }
    if (lane == 0) sh.red_i64[warp] = best, sh.red_int[warp] = best_idx;
    __syncthreads();
    if (warp == 0) {
        int64_t b = sh.red_i64[lane];
        int bi = sh.red_int[lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int64_t s2 = __shfl_xor_sync(0xFFFFFFFFu, b, o);
            const int i2 = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
            better(b, bi, s2, i2);
        }
        if (lane == 0) {
            unrank_partition(static_cast<uint32_t>(bi), n_parts, G, D, sh.h);
            sh.J = b;
        }
    }
    __syncthreads();
}

template <int DT>
__device__ void head_step(const Layer& L, Shared& sh, uint32_t n_parts) {
    head_sums<DT>(L, sh);
    choose_partition(L, sh, n_parts);
}

// ------------------------------------------------------------------ kernel --

template <int DT>
__global__ void __launch_bounds__(kThreads, 1)
search_kernel(const float* __restrict__ A_all, int G, int N, int D, int iters, int64_t n_parts,
              int32_t* __restrict__ head_out, int32_t* __restrict__ nu_out, int64_t* __restrict__ score_q_out,
              double* __restrict__ score_out, int32_t* __restrict__ iters_out, int* __restrict__ status_out,
              int* __restrict__ ws_status, uint8_t* __restrict__ gbuf, size_t per_layer, int use_smem) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ Shared sh;
    const int layer = blockIdx.x;
    uint8_t* buf = use_smem ? dsm : gbuf + static_cast<size_t>(layer) * per_layer;
    const float* A_glob = A_all + static_cast<int64_t>(layer) * G * N;
    Layer L;
    L.A = A_glob;
    L.G = G;
    L.N = N;
    L.D = D;
    L.cap = N / D;
    L.M = reinterpret_cast<int64_t*>(buf);
    L.nu = reinterpret_cast<int32_t*>(buf + static_cast<size_t>(N) * D * sizeof(int64_t));
    if (!use_smem) L.keys = reinterpret_cast<uint64_t*>(buf + mnu_bytes(N, D));
    if (use_smem == 2) {
        // A fits beside M and nu: copy it once; every pass then reads shared memory
        float* As = reinterpret_cast<float*>(buf + align_up_dev(static_cast<size_t>(N) * D * sizeof(int64_t) +
                                                                static_cast<size_t>(N) * sizeof(int32_t), 16));
        for_each_a(A_glob, static_cast<int64_t>(G) * N, [&](int64_t i, float a) { As[i] = a; });
        __syncthreads();
        L.A = As;
    }

    if (threadIdx.x == 0) {
        sh.status = DTP_OK;
        for (int l = 0; l < DMAX; ++l) sh.pi[l] = 0;
    }
    // validity and the fixed-point exponent
    uint32_t amax_bits = 0;
    int bad = 0;
    for_each_a(L.A, static_cast<int64_t>(G) * N, [&](int64_t, float a) {
        if (!(a >= 0.0f) || isinf(a)) bad = 1;
        else amax_bits = max(amax_bits, __float_as_uint(a));
    });
    bad = __syncthreads_or(bad);
    const int64_t amax_all = block_max_i64(static_cast<int64_t>(amax_bits), sh);
    if (bad) {
        if (threadIdx.x == 0) {
            status_out[layer] = DTP_ERR_ARG;
            atomicMin(ws_status, static_cast<int>(DTP_ERR_ARG));
        }
        return;
    }
    const float amax = __uint_as_float(static_cast<uint32_t>(amax_all));
    int e = 0;
    if (amax > 0.0f) frexpf(amax, &e);
    L.e = e;
    int64_t part = 0;
    for_each_a(L.A, static_cast<int64_t>(G) * N, [&](int64_t, float a) { part += quantize(a, e); });
    const int64_t total = block_sum_i64(part, sh);
    if (threadIdx.x < G) sh.h[threadIdx.x] = (threadIdx.x * D) / G;
    if (threadIdx.x == 0) sh.Jprev = -1;
    __syncthreads();

    int done = 0;
    for (int it = 0; it < iters; ++it) {
        build_gain<DT>(L, sh);
        if constexpr (DT == 2) neuron_step_d2(L, sh);
        else neuron_step_general<DT>(L, sh);
        if (sh.status != DTP_OK) break;
        head_step<DT>(L, sh, static_cast<uint32_t>(n_parts));
        done = it + 1;
        const bool stop = sh.J <= sh.Jprev;
        __syncthreads();
        if (threadIdx.x == 0) sh.Jprev = sh.J;
        __syncthreads();
        if (stop) break;
    }
    __syncthreads();
    if (sh.status != DTP_OK) {
        if (threadIdx.x == 0) {
            status_out[layer] = sh.status;
            atomicMin(ws_status, sh.status);
        }
        return;
    }
    for (int k = threadIdx.x; k < N; k += kThreads) nu_out[static_cast<int64_t>(layer) * N + k] = L.nu[k];
    if (threadIdx.x < G) head_out[static_cast<int64_t>(layer) * G + threadIdx.x] = sh.h[threadIdx.x];
    if (threadIdx.x == 0) {
        score_q_out[layer] = sh.J;
        score_out[layer] = total > 0 ? static_cast<double>(sh.J) / static_cast<double>(total) : 0.0;
        iters_out[layer] = done;
        status_out[layer] = DTP_OK;
    }
}

// ------------------------------------------------ global optimum (one layer) --
//
// J of one layer is unchanged when the device labels of h and nu are permuted
// together, so its maximum is the best exact neuron step over the UNLABELLED
// balanced head partitions, G!/((G/D)!^D D!) of them.  Each is taken in its
// canonical labelling (a label first appears after every smaller one), in
// lexicographic order; one block runs the exact neuron step of one (layer,
// partition) item, and a second kernel takes, per layer, the first partition
// with the largest value and recomputes its assignment.

__host__ __device__ inline uint64_t fact_u64(int n) {
    uint64_t f = 1;
    for (int i = 2; i <= n; ++i) f *= static_cast<uint64_t>(i);
    return f;
}

// Completions of a canonical prefix: r heads left, `used` labelled blocks with
// rem[] places left, D - used blocks not yet opened (cap places each, opened
// in order): r! / (prod rem! * cap!^(D-used) * (D-used)!).  r <= 16.
__device__ uint64_t rgs_completions(int r, const int* rem, int used, int D, int cap) {
    uint64_t n = fact_u64(r);
    for (int l = 0; l < used; ++l) n /= fact_u64(rem[l]);
    const int u = D - used;
    const uint64_t fc = fact_u64(cap);
    for (int i = 0; i < u; ++i) n /= fc;
    return n / fact_u64(u);
}

// The idx-th canonical balanced labelling in lexicographic order (thread-local).
__device__ bool unrank_canonical(uint64_t idx, int G, int D, int* h) {
    const int cap = G / D;
    int cnt[DMAX];
    for (int l = 0; l < DMAX; ++l) cnt[l] = 0;
    int used = 0;
    for (int k = 0; k < G; ++k) {
        bool placed = false;
        for (int l = 0; l <= used && l < D; ++l) {
            if (cnt[l] == cap) continue;
            ++cnt[l];
            const int used2 = l == used ? used + 1 : used;
            int rem[DMAX];
            for (int a = 0; a < used2; ++a) rem[a] = cap - cnt[a];
            const uint64_t c = rgs_completions(G - k - 1, rem, used2, D, cap);
            if (idx < c) {
                h[k] = l;
                used = used2;
                placed = true;
                break;
            }
            idx -= c;
            --cnt[l];
        }
        if (!placed) return false;
    }
    return true;
}

int64_t unlabelled_count(int G, int D) {
    const int cap = G / D;
    uint64_t n = fact_u64(G);
    for (int l = 0; l < D; ++l) n /= fact_u64(cap);
    return static_cast<int64_t>(n / fact_u64(D));
}

// Validity, the fixed-point exponent and the total of q of the layer in L.A.
__device__ bool layer_prologue(Layer& L, Shared& sh, int64_t* total_out) {
    const int64_t GN = static_cast<int64_t>(L.G) * L.N;
    uint32_t amax_bits = 0;
    int bad = 0;
    for_each_a(L.A, GN, [&](int64_t, float a) {
        if (!(a >= 0.0f) || isinf(a)) bad = 1;
        else amax_bits = max(amax_bits, __float_as_uint(a));
    });
    bad = __syncthreads_or(bad);
    const int64_t amax_all = block_max_i64(static_cast<int64_t>(amax_bits), sh);
    if (bad) return false;
    const float amax = __uint_as_float(static_cast<uint32_t>(amax_all));
    int e = 0;
    if (amax > 0.0f) frexpf(amax, &e);
    L.e = e;
    if (total_out) {
        int64_t part = 0;
        for_each_a(L.A, GN, [&](int64_t, float a) { part += quantize(a, e); });
        *total_out = block_sum_i64(part, sh);
    }
    return true;
}

// Layer view over the block's buffer (and an smem copy of A in mode 2).
__device__ void layer_view(Layer& L, const float* A_glob, int G, int N, int D, uint8_t* buf, int use_smem) {
    L.A = A_glob;
    L.G = G;
    L.N = N;
    L.D = D;
    L.cap = N / D;
    L.M = reinterpret_cast<int64_t*>(buf);
    L.nu = reinterpret_cast<int32_t*>(buf + static_cast<size_t>(N) * D * sizeof(int64_t));
    L.keys = use_smem ? nullptr : reinterpret_cast<uint64_t*>(buf + mnu_bytes(N, D));
    if (use_smem == 2) {
        float* As = reinterpret_cast<float*>(buf + align_up_dev(static_cast<size_t>(N) * D * sizeof(int64_t) +
                                                                static_cast<size_t>(N) * sizeof(int32_t), 16));
        for_each_a(A_glob, static_cast<int64_t>(G) * N, [&](int64_t i, float a) { As[i] = a; });
        __syncthreads();
        L.A = As;
    }
}

template <int DT>
__device__ int64_t assignment_value(const Layer& L, Shared& sh) {
    int64_t part = 0;
    for (int k = threadIdx.x; k < L.N; k += kThreads) part += L.M[static_cast<int64_t>(k) * DT + L.nu[k]];
    return block_sum_i64(part, sh);
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 1)
global_items_kernel(const float* __restrict__ A_all, int layers, int G, int N, int64_t n_unl,
                    int64_t* __restrict__ values, int* __restrict__ ws_status, uint8_t* __restrict__ gbuf,
                    size_t per_block, int use_smem) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ Shared sh;
    uint8_t* buf = use_smem ? dsm : gbuf + static_cast<size_t>(blockIdx.x) * per_block;
    const int64_t items = static_cast<int64_t>(layers) * n_unl;
    for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
        const int layer = static_cast<int>(item / n_unl);
        const int64_t pidx = item - static_cast<int64_t>(layer) * n_unl;
        Layer L;
        layer_view(L, A_all + static_cast<int64_t>(layer) * G * N, G, N, DT, buf, use_smem);
        if (threadIdx.x == 0) {
            sh.status = DTP_OK;
            for (int l = 0; l < DMAX; ++l) sh.pi[l] = 0;
            int hh[GMAX];
            if (!unrank_canonical(static_cast<uint64_t>(pidx), G, DT, hh)) sh.status = DTP_ERR_NOT_CONVERGED;
            for (int g = 0; g < G; ++g) sh.h[g] = hh[g];
        }
        if (!layer_prologue(L, sh, nullptr)) {
            if (threadIdx.x == 0) {
                values[item] = -1;
                atomicMin(ws_status, static_cast<int>(DTP_ERR_ARG));
            }
            __syncthreads();
            continue;
        }
        build_gain<DT>(L, sh);
        if constexpr (DT == 2) neuron_step_d2(L, sh);
        else neuron_step_general<DT>(L, sh);
        __syncthreads();
        if (sh.status != DTP_OK) {
            if (threadIdx.x == 0) {
                values[item] = -1;
                atomicMin(ws_status, sh.status);
            }
            __syncthreads();
            continue;
        }
        const int64_t v = assignment_value<DT>(L, sh);
        if (threadIdx.x == 0) values[item] = v;
        __syncthreads();
    }
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 1)
global_pick_kernel(const float* __restrict__ A_all, int G, int N, int64_t n_unl, const int64_t* __restrict__ values,
                   int32_t* __restrict__ head_out, int32_t* __restrict__ nu_out, int64_t* __restrict__ score_q_out,
                   double* __restrict__ score_out, int* __restrict__ ws_status, uint8_t* __restrict__ gbuf,
                   size_t per_block, int use_smem) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ Shared sh;
    const int layer = blockIdx.x;
    const int64_t* vals = values + static_cast<int64_t>(layer) * n_unl;
    // first index of the largest value (values < 0 mark failed items)
    int64_t best = -1;
    int best_idx = 0x7FFFFFFF;
    for (int64_t i = threadIdx.x; i < n_unl; i += kThreads) better(best, best_idx, vals[i], static_cast<int>(i));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const int64_t s2 = __shfl_xor_sync(0xFFFFFFFFu, best, o);
        const int i2 = __shfl_xor_sync(0xFFFFFFFFu, best_idx, o);
        better(best, best_idx, s2, i2);
    }
    if (lane == 0) sh.red_i64[warp] = best, sh.red_int[warp] = best_idx;
    __syncthreads();
    if (warp == 0) {
        int64_t b = sh.red_i64[lane];
        int bi = sh.red_int[lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int64_t s2 = __shfl_xor_sync(0xFFFFFFFFu, b, o);
            const int i2 = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
            better(b, bi, s2, i2);
        }
        if (lane == 0) {
            sh.J = b;
            sh.best_idx = bi;
        }
    }
    __syncthreads();
    if (sh.J < 0) {                                   // every item failed: already reported
        if (threadIdx.x == 0) atomicMin(ws_status, static_cast<int>(DTP_ERR_ARG));
        return;
    }
    uint8_t* buf = use_smem ? dsm : gbuf + static_cast<size_t>(blockIdx.x) * per_block;
    Layer L;
    layer_view(L, A_all + static_cast<int64_t>(layer) * G * N, G, N, DT, buf, use_smem);
    if (threadIdx.x == 0) {
        sh.status = DTP_OK;
        for (int l = 0; l < DMAX; ++l) sh.pi[l] = 0;
        int hh[GMAX];
        unrank_canonical(static_cast<uint64_t>(sh.best_idx), G, DT, hh);
        for (int g = 0; g < G; ++g) sh.h[g] = hh[g];
    }
    int64_t total = 0;
    layer_prologue(L, sh, &total);
    build_gain<DT>(L, sh);
    if constexpr (DT == 2) neuron_step_d2(L, sh);
    else neuron_step_general<DT>(L, sh);
    __syncthreads();
    if (sh.status != DTP_OK) {
        if (threadIdx.x == 0) atomicMin(ws_status, sh.status);
        return;
    }
    const int64_t v = assignment_value<DT>(L, sh);
    for (int k = threadIdx.x; k < N; k += kThreads) nu_out[static_cast<int64_t>(layer) * N + k] = L.nu[k];
    if (threadIdx.x < G) head_out[static_cast<int64_t>(layer) * G + threadIdx.x] = sh.h[threadIdx.x];
    if (threadIdx.x == 0) {
        score_q_out[layer] = v;
        score_out[layer] = total > 0 ? static_cast<double>(v) / static_cast<double>(total) : 0.0;
        if (v != sh.J) atomicMin(ws_status, static_cast<int>(DTP_ERR_NOT_CONVERGED));   // must recompute equal
    }
}

// ------------------------------------------------------- whole-model search --
//
// Eq. objective with both sums: J = sum_i up_i + sum_{i<L-1} down_i, each matrix
// in its exact unit-mass form n = floor(q 2^43 / total), q = floor(S 2^(40-e)),
// the product taken in 128 bits.  One
// iteration = every layer's neuron step given all head partitions (gain from
// h_i for the up edge and h_{i+1} for the down edge), then every layer's head
// step given all neuron assignments (column sums over nu_i for the up edge and
// nu_{i-1} for the down edge), then the score.  Each step maximises J exactly
// given the other block, so layers run in parallel, one block each.  A device
// flag stops later iterations after the first one (after the first) without a
// strict increase, so the host never waits.
//
// Ablations (Sec. 3 "Optimiser", Table 4): per-layer flags freeze a layer's
// heads or neurons at the contiguous start, and `minimize` minimises J.  A
// minimising step maximises R - gain with R the per-neuron (per-head) sum of
// the gains over devices: every neuron (head) sits on exactly one device, so
// the offset shifts all assignments' totals equally and leaves the set of
// optimal assignments (hence the canonical one) unchanged, while keeping every
// gain non-negative and below 2^44 as the exact steps require.

constexpr int kNormBits = 43;   // gains (one up + one down matrix) stay below 2^44
constexpr int kNormPreBits = 40;

struct ChainState {
    int done;
    int iters;
    int64_t prev;
};

__global__ void chain_init_kernel(ChainState* st, int64_t* J_q, double* J, int32_t* iters_done) {
    st->done = 0;
    st->iters = 0;
    st->prev = INT64_MIN;
    *J_q = 0;
    *J = 0.0;
    if (iters_done) *iters_done = 0;
}

// One block per matrix: m < L is the up edge of layer m, m >= L the down edge of layer m - L.
// head / nu (may be null) receive the contiguous start layout.
__global__ void __launch_bounds__(kThreads, 1)
chain_normalize_kernel(const float* __restrict__ S_up, const float* __restrict__ S_down, int L, int G, int N, int D,
                       int64_t* __restrict__ nbuf, int32_t* __restrict__ head, int32_t* __restrict__ nu,
                       ChainState* st, int* ws_status) {
    __shared__ Shared sh;
    const int m = blockIdx.x;
    const int64_t GN = static_cast<int64_t>(G) * N;
    const float* src = m < L ? S_up + m * GN : S_down + (m - L) * GN;
    int64_t* dst = nbuf + m * GN;
    if (m < L && head && threadIdx.x < G) head[m * G + threadIdx.x] = (threadIdx.x * D) / G;
    if (m < L && nu)
        for (int k = threadIdx.x; k < N; k += kThreads)
            nu[static_cast<int64_t>(m) * N + k] = static_cast<int>((static_cast<int64_t>(k) * D) / N);
    uint32_t amax_bits = 0;
    int bad = 0;
    for_each_a(src, GN, [&](int64_t, float a) {
        if (!(a >= 0.0f) || isinf(a)) bad = 1;
        else amax_bits = max(amax_bits, __float_as_uint(a));
    });
    bad = __syncthreads_or(bad);
    const int64_t amax_all = block_max_i64(static_cast<int64_t>(amax_bits), sh);
    if (bad) {
        if (threadIdx.x == 0) {
            atomicMin(ws_status, static_cast<int>(DTP_ERR_ARG));
            st->done = 1;
        }
        return;
    }
    const float amax = __uint_as_float(static_cast<uint32_t>(amax_all));
    int e = 0;
    if (amax > 0.0f) frexpf(amax, &e);
    int64_t part = 0;
    for_each_a(src, GN, [&](int64_t, float a) { part += quantize_bits(a, e, kNormPreBits); });
    const uint64_t total = static_cast<uint64_t>(block_sum_i64(part, sh));
    for_each_a(src, GN, [&](int64_t i, float a) {
        const uint64_t q = static_cast<uint64_t>(quantize_bits(a, e, kNormPreBits));
        dst[i] = total ? static_cast<int64_t>((static_cast<unsigned __int128>(q) << kNormBits) / total) : 0;
    });
}

// M[k,l] = up mass of k from heads of layer i on l + down mass of k into heads of layer i+1 on l;
// minimising: sum_l' M[k,l'] - M[k,l].
template <int DT>
__device__ void build_gain_chain(const Layer& L, Shared& sh, const int64_t* __restrict__ nU,
                                 const int64_t* __restrict__ nD, bool minimize) {
    for (int k = threadIdx.x; k < L.N; k += kThreads) {
        int64_t m[DT];
#pragma unroll
        for (int l = 0; l < DT; ++l) m[l] = 0;
        for (int g = 0; g < L.G; ++g) {
            const int64_t u = nU[static_cast<int64_t>(g) * L.N + k];
            const int64_t dn = nD ? nD[static_cast<int64_t>(g) * L.N + k] : 0;
            const int hg = sh.h[g], hn = nD ? sh.hn[g] : -1;
#pragma unroll
            for (int l = 0; l < DT; ++l) m[l] += (l == hg ? u : 0) + (l == hn ? dn : 0);
        }
        int64_t r = 0;
        if (minimize) {
#pragma unroll
            for (int l = 0; l < DT; ++l) r += m[l];
        }
#pragma unroll
        for (int l = 0; l < DT; ++l) L.M[static_cast<int64_t>(k) * DT + l] = minimize ? r - m[l] : m[l];
    }
    __syncthreads();
}

// B[g,l] = up mass of g on device l under nu_i + down mass into g from neurons of layer i-1 on l.
template <int DT>
__device__ void head_sums_chain(const Layer& L, Shared& sh, const int64_t* __restrict__ nU,
                                const int32_t* __restrict__ nu_i, const int64_t* __restrict__ nD,
                                const int32_t* __restrict__ nu_prev) {
    const int G = L.G;
    if (threadIdx.x < GMAX * DMAX) sh.B[threadIdx.x] = 0;
    __syncthreads();
    const int warps_per_head = kWarps / G;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = warp / warps_per_head;
    if (g < G) {
        const int tph = warps_per_head * 32;
        const int sub = (warp % warps_per_head) * 32 + lane;
        int64_t acc[DT];
#pragma unroll
        for (int l = 0; l < DT; ++l) acc[l] = 0;
        for (int k = sub; k < L.N; k += tph) {
            const int64_t u = nU[static_cast<int64_t>(g) * L.N + k];
            const int lu = nu_i[k];
            const int64_t dn = nD ? nD[static_cast<int64_t>(g) * L.N + k] : 0;
            const int ld = nD ? nu_prev[k] : -1;
#pragma unroll
            for (int l = 0; l < DT; ++l) acc[l] += (l == lu ? u : 0) + (l == ld ? dn : 0);
        }
#pragma unroll
        for (int l = 0; l < DT; ++l) {
            const int64_t v = warp_sum_i64(acc[l]);
            if (lane == 0 && v)
                atomicAdd(reinterpret_cast<unsigned long long*>(&sh.B[g * DT + l]), static_cast<unsigned long long>(v));
        }
    }
    __syncthreads();
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 1)
chain_neuron_kernel(int Lyr, int G, int N, const int64_t* __restrict__ nbuf, const int32_t* __restrict__ head,
                    int32_t* __restrict__ nu_out, int64_t* __restrict__ prices, ChainState* st, int* ws_status,
                    uint8_t* __restrict__ gbuf, size_t per_layer, int use_smem,
                    const uint8_t* __restrict__ move_neurons, int minimize) {
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ Shared sh;
    if (*reinterpret_cast<volatile int*>(&st->done)) return;
    const int i = blockIdx.x;
    if (move_neurons && !move_neurons[i]) return;   // frozen: nu_i stays contiguous
    const int64_t GN = static_cast<int64_t>(G) * N;
    uint8_t* buf = use_smem ? dsm : gbuf + static_cast<size_t>(i) * per_layer;
    Layer L;
    L.A = nullptr;
    L.G = G;
    L.N = N;
    L.D = DT;
    L.cap = N / DT;
    L.e = 0;
    L.M = reinterpret_cast<int64_t*>(buf);
    L.nu = reinterpret_cast<int32_t*>(buf + static_cast<size_t>(N) * DT * sizeof(int64_t));
    if (!use_smem) L.keys = reinterpret_cast<uint64_t*>(buf + mnu_bytes(N, DT));
    const bool has_down = i + 1 < Lyr;
    if (threadIdx.x < G) {
        sh.h[threadIdx.x] = head[i * G + threadIdx.x];
        sh.hn[threadIdx.x] = has_down ? head[(i + 1) * G + threadIdx.x] : -1;
    }
    if (threadIdx.x < DMAX) sh.pi[threadIdx.x] = prices[i * DMAX + threadIdx.x];
    if (threadIdx.x == 0) sh.status = DTP_OK;
    __syncthreads();
    build_gain_chain<DT>(L, sh, nbuf + i * GN, has_down ? nbuf + (Lyr + i) * GN : nullptr, minimize != 0);
    if constexpr (DT == 2) neuron_step_d2(L, sh);
    else neuron_step_general<DT>(L, sh);
    __syncthreads();
    if (sh.status != DTP_OK) {
        if (threadIdx.x == 0) {
            atomicMin(ws_status, sh.status);
            st->done = 1;
        }
        return;
    }
    for (int k = threadIdx.x; k < N; k += kThreads) nu_out[static_cast<int64_t>(i) * N + k] = L.nu[k];
    if (threadIdx.x < DMAX) prices[i * DMAX + threadIdx.x] = sh.pi[threadIdx.x];
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 1)
chain_head_kernel(int Lyr, int G, int N, const int64_t* __restrict__ nbuf, const int32_t* __restrict__ nu_all,
                  int32_t* __restrict__ head, int64_t* __restrict__ layer_score, ChainState* st, uint32_t n_parts,
                  const uint8_t* __restrict__ move_heads, int minimize) {
    __shared__ Shared sh;
    if (*reinterpret_cast<volatile int*>(&st->done)) return;
    const int i = blockIdx.x;
    const int64_t GN = static_cast<int64_t>(G) * N;
    Layer L;
    L.A = nullptr;
    L.G = G;
    L.N = N;
    L.D = DT;
    L.cap = N / DT;
    L.e = 0;
    L.M = nullptr;
    L.nu = nullptr;
    head_sums_chain<DT>(L, sh, nbuf + i * GN, nu_all + static_cast<int64_t>(i) * N,
                        i > 0 ? nbuf + (Lyr + i - 1) * GN : nullptr,
                        i > 0 ? nu_all + static_cast<int64_t>(i - 1) * N : nullptr);
    const int64_t sign = minimize ? -1 : 1;
    if (move_heads && !move_heads[i]) {            // frozen: score the current (contiguous) partition
        if (threadIdx.x == 0) {
            int64_t sc = 0;
            for (int g = 0; g < G; ++g) sc += sh.B[g * DT + head[i * G + g]];
            layer_score[i] = sign * sc;
        }
        return;
    }
    int64_t R = 0;                                  // sum_g R_g, held by thread 0
    if (minimize) {
        if (threadIdx.x < G) {
            int64_t r = 0;
#pragma unroll
            for (int l = 0; l < DT; ++l) r += sh.B[threadIdx.x * DT + l];
#pragma unroll
            for (int l = 0; l < DT; ++l) sh.B[threadIdx.x * DT + l] = r - sh.B[threadIdx.x * DT + l];
            sh.red_i64[threadIdx.x] = r;
        }
        __syncthreads();
        if (threadIdx.x == 0)
            for (int g = 0; g < G; ++g) R += sh.red_i64[g];
        __syncthreads();                            // choose_partition reuses red_i64
    }
    choose_partition(L, sh, n_parts);
    if (threadIdx.x < G) head[i * G + threadIdx.x] = sh.h[threadIdx.x];
    if (threadIdx.x == 0) layer_score[i] = sh.J - R;   // minimising: -(J of this layer) = J' - sum_g R_g
}

__global__ void chain_score_kernel(int Lyr, const int64_t* __restrict__ layer_score, ChainState* st, int64_t* J_q,
                                   double* J, int32_t* iters_done, int minimize) {
    if (threadIdx.x != 0 || st->done) return;
    int64_t total = 0;
    for (int i = 0; i < Lyr; ++i) total += layer_score[i];
    st->iters += 1;
    *iters_done = st->iters;
    const int64_t jq = minimize ? -total : total;
    *J_q = jq;
    *J = ldexp(static_cast<double>(jq), -kNormBits);
    if (total <= st->prev) st->done = 1;
    else st->prev = total;
}

// J of a given layout, per edge (Eq. objective): one block per edge, edge 2i =
// up_i (h_i(g) == nu_i(k)), edge 2i+1 = down_i (nu_i(k) == h_{i+1}(g)).
// Entries of h or nu outside [0, D) are reported as DTP_ERR_ARG.
__global__ void __launch_bounds__(kThreads, 1)
chain_edge_kernel(int Lyr, int G, int N, int D, const int64_t* __restrict__ nbuf, const int32_t* __restrict__ head,
                  const int32_t* __restrict__ nu, int64_t* __restrict__ edge, ChainState* st, int* ws_status) {
    __shared__ Shared sh;
    if (*reinterpret_cast<volatile int*>(&st->done)) return;
    const int e = blockIdx.x;
    const int i = e >> 1;
    const bool up = (e & 1) == 0;
    const int64_t GN = static_cast<int64_t>(G) * N;
    const int64_t* n = nbuf + (up ? i : Lyr + i) * GN;
    const int32_t* hg = head + static_cast<int64_t>(up ? i : i + 1) * G;
    const int32_t* nk = nu + static_cast<int64_t>(i) * N;
    if (threadIdx.x < G) sh.h[threadIdx.x] = hg[threadIdx.x];
    __syncthreads();
    int bad = 0;
    if (threadIdx.x < G && (sh.h[threadIdx.x] < 0 || sh.h[threadIdx.x] >= D)) bad = 1;
    int64_t part = 0;
    for (int k = threadIdx.x; k < N; k += kThreads) {
        const int l = nk[k];
        if (l < 0 || l >= D) {
            bad = 1;
            continue;
        }
        for (int g = 0; g < G; ++g)
            if (sh.h[g] == l) part += n[static_cast<int64_t>(g) * N + k];
    }
    bad = __syncthreads_or(bad);
    const int64_t tot = block_sum_i64(part, sh);
    if (threadIdx.x == 0) {
        edge[e] = tot;
        if (bad) atomicMin(ws_status, static_cast<int>(DTP_ERR_ARG));
    }
}

__global__ void chain_total_kernel(int n_edges, const int64_t* __restrict__ edge, const ChainState* st,
                                   int64_t* J_q, double* J) {
    if (threadIdx.x != 0 || st->done) return;
    int64_t t = 0;
    for (int e = 0; e < n_edges; ++e) t += edge[e];
    *J_q = t;
    *J = ldexp(static_cast<double>(t), -kNormBits);
}

// --------------------------------------------------------------------- host --

int64_t partition_count(int G, int D) {
    // G! / ((G/D)!)^D
    double f[GMAX + 1];
    f[0] = 1.0;
    for (int i = 1; i <= GMAX; ++i) f[i] = f[i - 1] * i;
    double c = f[G];
    for (int l = 0; l < D; ++l) c /= f[G / D];
    return static_cast<int64_t>(c + 0.5);
}

static size_t per_layer_bytes(int N, int D) {
    return align_up(static_cast<size_t>(N) * D * sizeof(int64_t) + static_cast<size_t>(N) * sizeof(int32_t), 256);
}

static bool fits_smem(int N, int D) { return per_layer_bytes(N, D) <= kSmemBudget; }

// bytes of M, nu and a copy of A [G,N] fp32 (the layout the kernel uses in mode 2)
static size_t with_a_bytes(int G, int N, int D) {
    return align_up(static_cast<size_t>(N) * D * sizeof(int64_t) + static_cast<size_t>(N) * sizeof(int32_t), 16) +
           static_cast<size_t>(G) * N * sizeof(float);
}

size_t workspace_bytes(int layers, int G, int N, int D) {
    (void)G;
    size_t b = kWorkspaceHeader + align_up(static_cast<size_t>(layers) * sizeof(int), 256);
    if (!fits_smem(N, D)) b += static_cast<size_t>(layers) * global_layer_bytes(N, D);
    return b;
}

int launch(const float* A, int layers, int G, int N, int D, int iters, int32_t* head, int32_t* nu, int64_t* score_q,
           double* score, int32_t* iters_done, void* workspace, cudaStream_t stream) {
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
    int* ws_status = reinterpret_cast<int*>(ws);
    int* status = reinterpret_cast<int*>(ws + kWorkspaceHeader);
    uint8_t* gbuf = ws + kWorkspaceHeader + align_up(static_cast<size_t>(layers) * sizeof(int), 256);
    const bool smem = fits_smem(N, D);
    const int mode = !smem ? 0 : (with_a_bytes(G, N, D) <= kSmemBudget ? 2 : 1);
    const size_t dyn = mode == 2 ? with_a_bytes(G, N, D) : (mode == 1 ? per_layer_bytes(N, D) : 0);
    void (*kernels[DMAX + 1])(const float*, int, int, int, int, int64_t, int32_t*, int32_t*, int64_t*, double*,
                              int32_t*, int*, int*, uint8_t*, size_t, int) = {
        nullptr, nullptr, search_kernel<2>, search_kernel<3>, search_kernel<4>,
        search_kernel<5>, search_kernel<6>, search_kernel<7>, search_kernel<8>};
    auto kern = kernels[D];
    DTP_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBudget)));
    // the header status word starts at DTP_OK; every block writes its layer's word
    DTP_CUDA_TRY(cudaMemsetAsync(ws_status, 0, kWorkspaceHeader, stream));
    kern<<<layers, kThreads, dyn, stream>>>(A, G, N, D, iters, partition_count(G, D), head, nu, score_q,
                                                      score, iters_done, status, ws_status, gbuf,
                                                      global_layer_bytes(N, D), mode);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace search
}  // namespace dtp

namespace dtp {
namespace search {

static size_t chain_layout(int Lyr, int G, int N, int D, size_t* off_state, size_t* off_score, size_t* off_prices,
                           size_t* off_nbuf, size_t* off_gbuf) {
    const size_t GN = static_cast<size_t>(G) * N;
    size_t o = kWorkspaceHeader;
    *off_state = o;
    o += 256;
    *off_score = o;
    o += align_up(static_cast<size_t>(2 * Lyr) * sizeof(int64_t), 256);   // layer scores / edge scores
    *off_prices = o;
    o += align_up(static_cast<size_t>(Lyr) * DMAX * sizeof(int64_t), 256);
    *off_nbuf = o;
    o += align_up(static_cast<size_t>(2 * Lyr - 1) * GN * sizeof(int64_t), 256);
    *off_gbuf = o;
    if (!fits_smem(N, D)) o += static_cast<size_t>(Lyr) * global_layer_bytes(N, D);
    return o;
}

size_t chain_workspace_bytes(int Lyr, int G, int N, int D) {
    size_t a, b, c, d, e;
    return chain_layout(Lyr, G, N, D, &a, &b, &c, &d, &e);
}

template <int DT>
static int launch_chain_t(const float* S_up, const float* S_down, int Lyr, int G, int N, int iters,
                          const uint8_t* move_heads, const uint8_t* move_neurons, int minimize, int32_t* head,
                          int32_t* nu, int64_t* J_q, double* J, int32_t* iters_done, uint8_t* ws,
                          cudaStream_t stream) {
    size_t o_state, o_score, o_prices, o_nbuf, o_gbuf;
    chain_layout(Lyr, G, N, DT, &o_state, &o_score, &o_prices, &o_nbuf, &o_gbuf);
    int* ws_status = reinterpret_cast<int*>(ws);
    ChainState* st = reinterpret_cast<ChainState*>(ws + o_state);
    int64_t* layer_score = reinterpret_cast<int64_t*>(ws + o_score);
    int64_t* prices = reinterpret_cast<int64_t*>(ws + o_prices);
    int64_t* nbuf = reinterpret_cast<int64_t*>(ws + o_nbuf);
    uint8_t* gbuf = ws + o_gbuf;
    const bool smem = fits_smem(N, DT);
    const size_t dyn = smem ? per_layer_bytes(N, DT) : 0;
    DTP_CUDA_TRY(cudaFuncSetAttribute(chain_neuron_kernel<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBudget)));
    DTP_CUDA_TRY(cudaMemsetAsync(ws_status, 0, kWorkspaceHeader, stream));
    DTP_CUDA_TRY(cudaMemsetAsync(prices, 0, static_cast<size_t>(Lyr) * DMAX * sizeof(int64_t), stream));
    chain_init_kernel<<<1, 1, 0, stream>>>(st, J_q, J, iters_done);
    chain_normalize_kernel<<<2 * Lyr - 1, kThreads, 0, stream>>>(S_up, S_down, Lyr, G, N, DT, nbuf, head, nu, st,
                                                                 ws_status);
    const uint32_t n_parts = static_cast<uint32_t>(partition_count(G, DT));
    for (int it = 0; it < iters; ++it) {
        chain_neuron_kernel<DT><<<Lyr, kThreads, dyn, stream>>>(Lyr, G, N, nbuf, head, nu, prices, st, ws_status, gbuf,
                                                                 global_layer_bytes(N, DT), smem ? 1 : 0, move_neurons,
                                                                 minimize);
        chain_head_kernel<DT><<<Lyr, kThreads, 0, stream>>>(Lyr, G, N, nbuf, nu, head, layer_score, st, n_parts,
                                                             move_heads, minimize);
        chain_score_kernel<<<1, 32, 0, stream>>>(Lyr, layer_score, st, J_q, J, iters_done, minimize);
    }
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

int launch_chain(const float* S_up, const float* S_down, int Lyr, int G, int N, int D, int iters,
                 const uint8_t* move_heads, const uint8_t* move_neurons, int minimize, int32_t* head, int32_t* nu,
                 int64_t* J_q, double* J, int32_t* iters_done, void* workspace, cudaStream_t stream) {
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
#define DTP_CHAIN_CASE(DV)                                                                                  \
    case DV:                                                                                                \
        return launch_chain_t<DV>(S_up, S_down, Lyr, G, N, iters, move_heads, move_neurons, minimize, head, nu, \
                                  J_q, J, iters_done, ws, stream);
    switch (D) {
        DTP_CHAIN_CASE(2)
        DTP_CHAIN_CASE(3)
        DTP_CHAIN_CASE(4)
        DTP_CHAIN_CASE(5)
        DTP_CHAIN_CASE(6)
        DTP_CHAIN_CASE(7)
        DTP_CHAIN_CASE(8)
        default: return DTP_ERR_ARG;
    }
#undef DTP_CHAIN_CASE
}

static size_t global_layout_bytes(int layers, int G, int N, int D, int grid, size_t* off_vals, size_t* off_gbuf) {
    size_t o = kWorkspaceHeader;
    *off_vals = o;
    o += align_up(static_cast<size_t>(layers) * unlabelled_count(G, D) * sizeof(int64_t), 256);
    *off_gbuf = o;
    if (!fits_smem(N, D)) o += static_cast<size_t>(grid > layers ? grid : layers) * global_layer_bytes(N, D);
    return o;
}

// The item kernel's grid: one block per SM, at most kGlobalMaxGrid (the workspace holds a
// per-block buffer for that many blocks when the layer does not fit in shared memory).
constexpr int kGlobalMaxGrid = 160;

static int global_grid(int layers, int G, int D) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev))
        return -1;
    if (sms > kGlobalMaxGrid) sms = kGlobalMaxGrid;
    const int64_t items = static_cast<int64_t>(layers) * unlabelled_count(G, D);
    return static_cast<int>(items < sms ? items : sms);
}

size_t global_workspace_bytes(int layers, int G, int N, int D) {
    size_t a, b;
    return global_layout_bytes(layers, G, N, D, kGlobalMaxGrid, &a, &b);
}

template <int DT>
static int launch_global_t(const float* A, int layers, int G, int N, int32_t* head, int32_t* nu, int64_t* score_q,
                           double* score, uint8_t* ws, cudaStream_t stream) {
    const int grid = global_grid(layers, G, DT);
    if (grid <= 0) return DTP_ERR_CUDA;
    size_t o_vals, o_gbuf;
    global_layout_bytes(layers, G, N, DT, grid, &o_vals, &o_gbuf);
    int* ws_status = reinterpret_cast<int*>(ws);
    int64_t* vals = reinterpret_cast<int64_t*>(ws + o_vals);
    uint8_t* gbuf = ws + o_gbuf;
    const bool smem = fits_smem(N, DT);
    const int mode = !smem ? 0 : (with_a_bytes(G, N, DT) <= kSmemBudget ? 2 : 1);
    const size_t dyn = mode == 2 ? with_a_bytes(G, N, DT) : (mode == 1 ? per_layer_bytes(N, DT) : 0);
    const int64_t n_unl = unlabelled_count(G, DT);
    DTP_CUDA_TRY(cudaFuncSetAttribute(global_items_kernel<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBudget)));
    DTP_CUDA_TRY(cudaFuncSetAttribute(global_pick_kernel<DT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      static_cast<int>(kSmemBudget)));
    DTP_CUDA_TRY(cudaMemsetAsync(ws_status, 0, kWorkspaceHeader, stream));
    global_items_kernel<DT><<<grid, kThreads, dyn, stream>>>(A, layers, G, N, n_unl, vals, ws_status, gbuf,
                                                             global_layer_bytes(N, DT), mode);
    global_pick_kernel<DT><<<layers, kThreads, dyn, stream>>>(A, G, N, n_unl, vals, head, nu, score_q, score,
                                                              ws_status, gbuf, global_layer_bytes(N, DT), mode);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

int launch_global(const float* A, int layers, int G, int N, int D, int32_t* head, int32_t* nu, int64_t* score_q,
                  double* score, void* workspace, cudaStream_t stream) {
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
    switch (D) {
        case 2: return launch_global_t<2>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 3: return launch_global_t<3>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 4: return launch_global_t<4>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 5: return launch_global_t<5>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 6: return launch_global_t<6>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 7: return launch_global_t<7>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        case 8: return launch_global_t<8>(A, layers, G, N, head, nu, score_q, score, ws, stream);
        default: return DTP_ERR_ARG;
    }
}

int launch_chain_score(const float* S_up, const float* S_down, int Lyr, int G, int N, int D, const int32_t* head,
                       const int32_t* nu, int64_t* edge_q, int64_t* J_q, double* J, void* workspace,
                       cudaStream_t stream) {
    uint8_t* ws = reinterpret_cast<uint8_t*>(workspace);
    size_t o_state, o_score, o_prices, o_nbuf, o_gbuf;
    chain_layout(Lyr, G, N, D, &o_state, &o_score, &o_prices, &o_nbuf, &o_gbuf);
    int* ws_status = reinterpret_cast<int*>(ws);
    ChainState* st = reinterpret_cast<ChainState*>(ws + o_state);
    int64_t* edge = edge_q ? edge_q : reinterpret_cast<int64_t*>(ws + o_score);
    int64_t* nbuf = reinterpret_cast<int64_t*>(ws + o_nbuf);
    DTP_CUDA_TRY(cudaMemsetAsync(ws_status, 0, kWorkspaceHeader, stream));
    chain_init_kernel<<<1, 1, 0, stream>>>(st, J_q, J, nullptr);
    chain_normalize_kernel<<<2 * Lyr - 1, kThreads, 0, stream>>>(S_up, S_down, Lyr, G, N, D, nbuf, nullptr, nullptr,
                                                                 st, ws_status);
    chain_edge_kernel<<<2 * Lyr - 1, kThreads, 0, stream>>>(Lyr, G, N, D, nbuf, head, nu, edge, st, ws_status);
    chain_total_kernel<<<1, 32, 0, stream>>>(2 * Lyr - 1, edge, st, J_q, J);
    DTP_CUDA_TRY(cudaGetLastError());
    return DTP_OK;
}

}  // namespace search
}  // namespace dtp
