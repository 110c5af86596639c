// dtp_api.cu -- the extern "C" entry points declared in include/dtp.h:
// argument validation on the host, then dispatch to the kernels.
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace dtp {
namespace tc {
size_t workspace_bytes(int64_t T, int d, int G, int N);
size_t workspace_bytes_with_act(int64_t T, int d, int G, int N);
int launch(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A,
           void* workspace, cudaStream_t stream, const float* rms, float* act2);
int launch_grouped(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N,
                   float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2, int qpg,
                   int max_ctas, int defer_reduce);
int launch_reduce(const void* workspace, int64_t T, int d, int G, int N, float* A, float* act2, int qpg,
                  cudaStream_t stream, int max_blocks, int overwrite);
}  // namespace tc
namespace f32 {
size_t workspace_bytes(int64_t T, int d, int G, int N);
int launch(const float* X, const float* C, const float* Wg, const float* Wu, int64_t T, int d, int G, int N,
           float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2);
int launch_grouped(const float* X, const float* C, const float* Wg, const float* Wu, int64_t T, int d, int G, int N,
                   float* A, void* workspace, cudaStream_t stream, const float* rms, float* act2, int qpg);
}  // namespace f32
namespace sq {
size_t down_workspace_bytes(int G, int R, int d, int N);
int launch_down(const void* Wqkv, const void* gamma, const void* Wd, int G, int R, int d, int N, int dtype, float* bn,
                void* workspace, cudaStream_t stream);
size_t add_workspace_bytes(int64_t T, int G, int N);
int launch_add(const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A_add,
               void* workspace, cudaStream_t stream);
int launch_add_grouped(const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A_add,
                       void* workspace, cudaStream_t stream, int qpg);
}  // namespace sq
namespace hw {
int launch(const void* attn, const void* Wo, const float* gamma, const float* rms, int64_t T, int d, int Hq, int hd,
           int q_per_row, void* C, void* workspace, cudaStream_t stream);
}  // namespace hw
namespace apply {
int launch_order(const int32_t* labels, int layers, int n, int D, int balanced, int32_t* order, void* workspace,
                 cudaStream_t stream);
int launch_rows(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int block_rows,
                const int32_t* perm, int64_t perm_stride, void* workspace, cudaStream_t stream);
int launch_cols(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int64_t block_bytes,
                int elem_bytes, const int32_t* perm, int64_t perm_stride, void* workspace, cudaStream_t stream);
}  // namespace apply
int launch_finalize(float* A, int G, int N, int64_t T_total, const float* wd, cudaStream_t stream);
int launch_top_share(const float* A, int layers, int G, int N, double* share, cudaStream_t stream);
int launch_down_finalize(const float* act2, const float* bn, int G, int N, int64_t T_total, float* S,
                         cudaStream_t stream);
int launch_down_sqnorm(const void* W, int d, int N, int dtype, float* out, cudaStream_t stream);
namespace search {
size_t workspace_bytes(int layers, int G, int N, int D);
int64_t partition_count(int G, int D);
int launch(const float* A, int layers, int G, int N, int D, int iters, int32_t* head, int32_t* nu, int64_t* score_q,
           double* score, int32_t* iters_done, void* workspace, cudaStream_t stream);
size_t chain_workspace_bytes(int Lyr, int G, int N, int D);
int64_t unlabelled_count(int G, int D);
size_t global_workspace_bytes(int layers, int G, int N, int D);
int launch_global(const float* A, int layers, int G, int N, int D, int32_t* head, int32_t* nu, int64_t* score_q,
                  double* score, void* workspace, cudaStream_t stream);
int launch_chain(const float* S_up, const float* S_down, int Lyr, int G, int N, int D, int iters,
                 const uint8_t* move_heads, const uint8_t* move_neurons, int minimize, int32_t* head, int32_t* nu,
                 int64_t* J_q, double* J, int32_t* iters_done, void* workspace, cudaStream_t stream);
int launch_chain_score(const float* S_up, const float* S_down, int Lyr, int G, int N, int D, const int32_t* head,
                       const int32_t* nu, int64_t* edge_q, int64_t* J_q, double* J, void* workspace,
                       cudaStream_t stream);
}  // namespace search
}  // namespace dtp

using namespace dtp;

namespace {

constexpr int kMaxHeads = 16;

bool affinity_sizes_ok(int64_t T, int d, int H, int N, int dtype) {
    if (dtype != DTP_BF16 && dtype != DTP_F32) return false;
    if (T < 0 || d < 8 || (d % 8) != 0 || H < 1 || H > kMaxHeads || N < 1) return false;
    // TMA coordinates are int32 and the token axis of C is addressed in one box dimension
    if (T > (int64_t(1) << 31) - 256 || N > (1 << 30)) return false;
    return true;
}

size_t affinity_ws(int64_t T, int d, int H, int N, int dtype, bool with_act) {
    if (dtype != DTP_BF16) return f32::workspace_bytes(T, d, H, N);
    return with_act ? tc::workspace_bytes_with_act(T, d, H, N) : tc::workspace_bytes(T, d, H, N);
}

// Query heads per launch of the grouped affinity: the largest multiple of qpg within kMaxHeads.
constexpr int kMaxQueryHeads = 128;
int grouped_chunk(int H_q, int qpg) {
    const int c = (kMaxHeads / qpg) * qpg;
    return H_q < c ? H_q : c;
}

bool grouped_sizes_ok(int64_t T, int d, int H_q, int qpg, int N, int dtype) {
    if (qpg < 1 || qpg > kMaxHeads || H_q < 1 || H_q > kMaxQueryHeads || H_q % qpg || H_q / qpg > kMaxHeads)
        return false;
    return affinity_sizes_ok(T, d, grouped_chunk(H_q, qpg), N, dtype);
}

bool search_sizes_ok(int layers, int H, int N, int D, int iters) {
    if (layers < 1 || D < 2 || D > 8 || H < 1 || H > kMaxHeads || N < 1 || iters < 1) return false;
    if (H % D || N % D) return false;
    if (N > (1 << 18) || static_cast<int64_t>(H) * N > (int64_t(1) << 22)) return false;
    if (search::partition_count(H, D) > (int64_t(1) << 26)) return false;
    return true;
}

}  // namespace

extern "C" {

int dtp_version(void) { return 100; }

const char* dtp_status_string(int status) {
    switch (status) {
        case DTP_OK: return "ok";
        case DTP_ERR_ARG: return "invalid argument";
        case DTP_ERR_CUDA: return "CUDA error";
        case DTP_ERR_NOT_CONVERGED: return "bounded device loop or wait hit its limit";
        case DTP_ERR_UNSUPPORTED: return "unsupported";
        case DTP_ERR_WORKSPACE: return "workspace missing or too small";
        default: return "unknown status";
    }
}

int dtp_affinity_workspace_size(int64_t T, int d, int H_kv, int N, int dtype, size_t* bytes) {
    if (!bytes || !affinity_sizes_ok(T, d, H_kv, N, dtype)) return DTP_ERR_ARG;
    *bytes = affinity_ws(T, d, H_kv, N, dtype, true);
    return DTP_OK;
}

int dtp_affinity_accumulate_ex(const void* X, const void* C, const void* W_gate, const void* W_up,
                               const float* rms_next, int64_t T, int d, int H_kv, int N, int dtype, float* A,
                               float* act2, void* workspace, size_t workspace_bytes, void* stream) {
    if (!affinity_sizes_ok(T, d, H_kv, N, dtype)) return DTP_ERR_ARG;
    if ((rms_next == nullptr) != (act2 == nullptr)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;  // nothing to add; empty inputs may have null data pointers
    if (!X || !C || !W_gate || !W_up || !A) return DTP_ERR_ARG;
    if (!aligned16(X) || !aligned16(C) || !aligned16(W_gate) || !aligned16(W_up) || !aligned16(A))
        return DTP_ERR_ARG;
    const bool with_act = act2 != nullptr;
    if (with_act && (!aligned16(act2) || !aligned16(rms_next))) return DTP_ERR_ARG;
    const size_t need = affinity_ws(T, d, H_kv, N, dtype, with_act);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    if (dtype == DTP_BF16) return tc::launch(X, C, W_gate, W_up, T, d, H_kv, N, A, workspace, s, rms_next, act2);
    return f32::launch(static_cast<const float*>(X), static_cast<const float*>(C), static_cast<const float*>(W_gate),
                       static_cast<const float*>(W_up), T, d, H_kv, N, A, workspace, s, rms_next, act2);
}

int dtp_affinity_accumulate_opts(const void* X, const void* C, const void* W_gate, const void* W_up,
                                 const float* rms_next, int64_t T, int d, int H_kv, int N, int dtype, float* A,
                                 float* act2, const dtp_affinity_opts* opts, void* workspace, size_t workspace_bytes,
                                 void* stream) {
    if (!opts || opts->max_ctas < 0 || (opts->flags & ~DTP_AFFINITY_DEFER_REDUCE)) return DTP_ERR_ARG;
    for (int i = 0; i < 6; ++i)
        if (opts->reserved[i] != 0) return DTP_ERR_ARG;
    const int defer = (opts->flags & DTP_AFFINITY_DEFER_REDUCE) != 0;
    if (defer && dtype != DTP_BF16) return DTP_ERR_UNSUPPORTED;
    if (dtype != DTP_BF16 || (opts->max_ctas == 0 && !defer))
        return dtp_affinity_accumulate_ex(X, C, W_gate, W_up, rms_next, T, d, H_kv, N, dtype, A, act2, workspace,
                                          workspace_bytes, stream);
    if (!affinity_sizes_ok(T, d, H_kv, N, dtype)) return DTP_ERR_ARG;
    if ((rms_next == nullptr) != (act2 == nullptr)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!X || !C || !W_gate || !W_up || !A) return DTP_ERR_ARG;
    if (!aligned16(X) || !aligned16(C) || !aligned16(W_gate) || !aligned16(W_up) || !aligned16(A))
        return DTP_ERR_ARG;
    const bool with_act = act2 != nullptr;
    if (with_act && (!aligned16(act2) || !aligned16(rms_next))) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < affinity_ws(T, d, H_kv, N, dtype, with_act) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return tc::launch_grouped(X, C, W_gate, W_up, T, d, H_kv, N, A, workspace, s, rms_next, act2, 1, opts->max_ctas,
                              defer);
}

int dtp_affinity_reduce(const void* workspace, size_t workspace_bytes, int64_t T, int d, int H_kv, int N, float* A,
                        float* act2, int max_blocks, int overwrite, void* stream) {
    if (!affinity_sizes_ok(T, d, H_kv, N, DTP_BF16) || max_blocks < 0 || max_blocks > 65535) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!A || !aligned16(A) || (act2 && !aligned16(act2))) return DTP_ERR_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < affinity_ws(T, d, H_kv, N, DTP_BF16, act2 != nullptr))
        return DTP_ERR_WORKSPACE;
    return tc::launch_reduce(workspace, T, d, H_kv, N, A, act2, 1, static_cast<cudaStream_t>(stream), max_blocks,
                             overwrite ? 1 : 0);
}

int dtp_affinity_accumulate(const void* X, const void* C, const void* W_gate, const void* W_up, int64_t T, int d,
                            int H_kv, int N, int dtype, float* A, void* workspace, size_t workspace_bytes,
                            void* stream) {
    return dtp_affinity_accumulate_ex(X, C, W_gate, W_up, nullptr, T, d, H_kv, N, dtype, A, nullptr, workspace,
                                      workspace_bytes, stream);
}

int dtp_affinity_grouped_workspace_size(int64_t T, int d, int H_q, int q_per_group, int N, int dtype,
                                        size_t* bytes) {
    if (!bytes || !grouped_sizes_ok(T, d, H_q, q_per_group, N, dtype)) return DTP_ERR_ARG;
    *bytes = affinity_ws(T, d, grouped_chunk(H_q, q_per_group), N, dtype, true);
    return DTP_OK;
}

int dtp_affinity_accumulate_grouped(const void* X, const void* C_q, const void* W_gate, const void* W_up,
                                    const float* rms_next, int64_t T, int d, int H_q, int q_per_group, int N,
                                    int dtype, float* A, float* act2, void* workspace, size_t workspace_bytes,
                                    void* stream) {
    if (!grouped_sizes_ok(T, d, H_q, q_per_group, N, dtype)) return DTP_ERR_ARG;
    if ((rms_next == nullptr) != (act2 == nullptr)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!X || !C_q || !W_gate || !W_up || !A) return DTP_ERR_ARG;
    if (!aligned16(X) || !aligned16(C_q) || !aligned16(W_gate) || !aligned16(W_up) || !aligned16(A))
        return DTP_ERR_ARG;
    const bool with_act = act2 != nullptr;
    if (with_act && (!aligned16(act2) || !aligned16(rms_next))) return DTP_ERR_ARG;
    const int chunk = grouped_chunk(H_q, q_per_group);
    const size_t need = affinity_ws(T, d, chunk, N, dtype, with_act);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    const size_t elem = dtype == DTP_BF16 ? 2 : 4;
    // chunks of whole KV groups; each chunk's C block starts 16-byte aligned (d % 8 == 0)
    for (int h0 = 0; h0 < H_q; h0 += chunk) {
        const int hc = H_q - h0 < chunk ? H_q - h0 : chunk;
        const void* Cc = static_cast<const uint8_t*>(C_q) + static_cast<size_t>(h0) * T * d * elem;
        float* Ac = A + static_cast<int64_t>(h0 / q_per_group) * N;
        const float* r = h0 == 0 ? rms_next : nullptr;   // the activation term once, with the first chunk
        float* a2 = h0 == 0 ? act2 : nullptr;
        const int st = dtype == DTP_BF16
                           ? tc::launch_grouped(X, Cc, W_gate, W_up, T, d, hc, N, Ac, workspace, s, r, a2, q_per_group,
                                                0, 0)
                           : f32::launch_grouped(static_cast<const float*>(X), static_cast<const float*>(Cc),
                                                 static_cast<const float*>(W_gate), static_cast<const float*>(W_up), T,
                                                 d, hc, N, Ac, workspace, s, r, a2, q_per_group);
        if (st != DTP_OK) return st;
    }
    return DTP_OK;
}

int dtp_affinity_add_workspace_size(int64_t T, int d, int H_kv, int N, size_t* bytes) {
    if (!bytes || !affinity_sizes_ok(T, d, H_kv, N, DTP_BF16)) return DTP_ERR_ARG;
    *bytes = sq::add_workspace_bytes(T, H_kv, N);
    return DTP_OK;
}

int dtp_affinity_add_accumulate(const void* C, const void* W_gate, const void* W_up, int64_t T, int d, int H_kv,
                                int N, float* A_add, void* workspace, size_t workspace_bytes, void* stream) {
    if (!affinity_sizes_ok(T, d, H_kv, N, DTP_BF16)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!C || !W_gate || !W_up || !A_add || !aligned16(C) || !aligned16(W_gate) || !aligned16(W_up) ||
        !aligned16(A_add))
        return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < sq::add_workspace_bytes(T, H_kv, N) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return sq::launch_add(C, W_gate, W_up, T, d, H_kv, N, A_add, workspace, s);
}

int dtp_affinity_add_grouped_workspace_size(int64_t T, int d, int H_q, int q_per_group, int N, size_t* bytes) {
    if (!bytes || !grouped_sizes_ok(T, d, H_q, q_per_group, N, DTP_BF16)) return DTP_ERR_ARG;
    *bytes = sq::add_workspace_bytes(T, grouped_chunk(H_q, q_per_group), N);
    return DTP_OK;
}

int dtp_affinity_add_accumulate_grouped(const void* C_q, const void* W_gate, const void* W_up, int64_t T, int d,
                                        int H_q, int q_per_group, int N, float* A_add, void* workspace,
                                        size_t workspace_bytes, void* stream) {
    if (!grouped_sizes_ok(T, d, H_q, q_per_group, N, DTP_BF16)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!C_q || !W_gate || !W_up || !A_add || !aligned16(C_q) || !aligned16(W_gate) || !aligned16(W_up) ||
        !aligned16(A_add))
        return DTP_ERR_ARG;
    const int chunk = grouped_chunk(H_q, q_per_group);
    if (!workspace || workspace_bytes < sq::add_workspace_bytes(T, chunk, N) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    for (int h0 = 0; h0 < H_q; h0 += chunk) {
        const int hc = H_q - h0 < chunk ? H_q - h0 : chunk;
        const void* Cc = static_cast<const uint8_t*>(C_q) + static_cast<size_t>(h0) * T * d * 2;
        const int st = sq::launch_add_grouped(Cc, W_gate, W_up, T, d, hc, N, A_add + static_cast<int64_t>(h0 / q_per_group) * N,
                                              workspace, s, q_per_group);
        if (st != DTP_OK) return st;
    }
    return DTP_OK;
}

int dtp_head_writes_workspace_size(size_t* bytes) {
    if (!bytes) return DTP_ERR_ARG;
    *bytes = kWorkspaceHeader;
    return DTP_OK;
}

int dtp_head_writes(const void* attn, const void* W_o, const float* gamma, const float* rms, int64_t T, int d,
                    int H_q, int head_dim, int q_per_row, void* C, void* workspace, size_t workspace_bytes,
                    void* stream) {
    if (T < 0 || T > (int64_t(1) << 31) - 256 || d < 8 || d % 8 || H_q < 1 || head_dim < 16 || head_dim % 16 ||
        q_per_row < 1 || H_q % q_per_row || static_cast<int64_t>(H_q) * head_dim > (int64_t(1) << 20) ||
        H_q / q_per_row > 65535)
        return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!attn || !W_o || !gamma || !rms || !C || !aligned16(attn) || !aligned16(W_o) || !aligned16(gamma) ||
        !aligned16(C) || (reinterpret_cast<uintptr_t>(rms) & 3))
        return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < kWorkspaceHeader || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return hw::launch(attn, W_o, gamma, rms, T, d, H_q, head_dim, q_per_row, C, workspace, s);
}

int dtp_layout_order(const int32_t* labels, int layers, int n, int D, int balanced, int32_t* order, void* workspace,
                     size_t workspace_bytes, void* stream) {
    if (layers < 1 || layers > 65535 || n < 1 || D < 1 || D > n || (balanced && n % D)) return DTP_ERR_ARG;
    if (!labels || !order || (reinterpret_cast<uintptr_t>(labels) & 3) || (reinterpret_cast<uintptr_t>(order) & 3))
        return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < kWorkspaceHeader || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return apply::launch_order(labels, layers, n, D, balanced ? 1 : 0, order, workspace, s);
}

int dtp_permute_rows(const void* src, void* dst, int layers, int64_t rows, int64_t row_bytes, int block_rows,
                     const int32_t* perm, int64_t perm_layer_stride, void* workspace, size_t workspace_bytes,
                     void* stream) {
    if (layers < 1 || rows < 1 || row_bytes < 1 || block_rows < 1 || rows % block_rows ||
        perm_layer_stride < rows / block_rows)
        return DTP_ERR_ARG;
    if (!src || !dst || !perm || src == dst || (reinterpret_cast<uintptr_t>(perm) & 3)) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < kWorkspaceHeader || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return apply::launch_rows(src, dst, layers, rows, row_bytes, block_rows, perm, perm_layer_stride, workspace, s);
}

int dtp_permute_cols(const void* src, void* dst, int layers, int64_t rows, int64_t cols, int elem_bytes,
                     int block_cols, const int32_t* perm, int64_t perm_layer_stride, void* workspace,
                     size_t workspace_bytes, void* stream) {
    if (layers < 1 || rows < 1 || cols < 1 || elem_bytes < 1 || elem_bytes > 16 || block_cols < 1 ||
        cols % block_cols || perm_layer_stride < cols / block_cols || cols * elem_bytes >= (int64_t(1) << 31))
        return DTP_ERR_ARG;
    if (!src || !dst || !perm || src == dst || (reinterpret_cast<uintptr_t>(perm) & 3)) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < kWorkspaceHeader || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return apply::launch_cols(src, dst, layers, rows, cols * elem_bytes, static_cast<int64_t>(block_cols) * elem_bytes,
                              elem_bytes, perm, perm_layer_stride, workspace, s);
}

int dtp_apply_layout(const int32_t* head_part, const int32_t* neuron_dev, int layers, int H_kv, int N, int D,
                     int q_per_group, int head_dim, int d, int elem_bytes, const void* const* src, void* const* dst,
                     int32_t* head_order, int32_t* neuron_order, void* workspace, size_t workspace_bytes,
                     void* stream) {
    if (layers < 1 || layers > 65535 || H_kv < 1 || N < 1 || D < 1 || H_kv % D || N % D || q_per_group < 1 ||
        head_dim < 1 || d < 1 || elem_bytes < 1 || elem_bytes > 16)
        return DTP_ERR_ARG;
    if (!head_part || !neuron_dev || !src || !dst || !head_order || !neuron_order) return DTP_ERR_ARG;
    for (int i = 0; i < 7; ++i)
        if (!src[i] || !dst[i] || src[i] == dst[i]) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < kWorkspaceHeader || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    int st = apply::launch_order(head_part, layers, H_kv, D, 1, head_order, workspace, s);
    if (st == DTP_OK) st = apply::launch_order(neuron_dev, layers, N, D, 1, neuron_order, workspace, s);
    const int64_t qrows = static_cast<int64_t>(H_kv) * q_per_group * head_dim;   // q_proj rows, o_proj columns
    const int64_t kvrows = static_cast<int64_t>(H_kv) * head_dim;
    const int64_t row = static_cast<int64_t>(d) * elem_bytes;
    const int qblk = q_per_group * head_dim;
    // q, k, v rows and o columns by KV group; gate, up rows and down columns by neuron
    if (st == DTP_OK) st = apply::launch_rows(src[0], dst[0], layers, qrows, row, qblk, head_order, H_kv, workspace, s);
    if (st == DTP_OK) st = apply::launch_rows(src[1], dst[1], layers, kvrows, row, head_dim, head_order, H_kv, workspace, s);
    if (st == DTP_OK) st = apply::launch_rows(src[2], dst[2], layers, kvrows, row, head_dim, head_order, H_kv, workspace, s);
    if (st == DTP_OK)
        st = apply::launch_cols(src[3], dst[3], layers, d, qrows * elem_bytes, static_cast<int64_t>(qblk) * elem_bytes,
                                elem_bytes, head_order, H_kv, workspace, s);
    if (st == DTP_OK) st = apply::launch_rows(src[4], dst[4], layers, N, row, 1, neuron_order, N, workspace, s);
    if (st == DTP_OK) st = apply::launch_rows(src[5], dst[5], layers, N, row, 1, neuron_order, N, workspace, s);
    if (st == DTP_OK)
        st = apply::launch_cols(src[6], dst[6], layers, d, static_cast<int64_t>(N) * elem_bytes, elem_bytes,
                                elem_bytes, neuron_order, N, workspace, s);
    return st;
}

int dtp_affinity_top_share(const float* A, int layers, int H_kv, int N, double* share, void* stream) {
    if (layers < 1 || layers > 65535 || H_kv < 1 || H_kv > kMaxHeads || N < 1) return DTP_ERR_ARG;
    if (!A || !share || (reinterpret_cast<uintptr_t>(A) & 3) || (reinterpret_cast<uintptr_t>(share) & 7))
        return DTP_ERR_ARG;
    return launch_top_share(A, layers, H_kv, N, share, static_cast<cudaStream_t>(stream));
}

int dtp_down_weight_workspace_size(int H_kv, int R, int d, int N, size_t* bytes) {
    if (!bytes || H_kv < 1 || H_kv > kMaxHeads || R < 1 || d < 8 || (d % 8) || N < 1) return DTP_ERR_ARG;
    *bytes = sq::down_workspace_bytes(H_kv, R, d, N);
    return DTP_OK;
}

int dtp_down_weight_sqnorm(const void* Wqkv_next, const void* gamma_next, const void* W_down, int H_kv, int R, int d,
                           int N, int dtype, float* bn, void* workspace, size_t workspace_bytes, void* stream) {
    if (H_kv < 1 || H_kv > kMaxHeads || R < 1 || d < 8 || (d % 8) || N < 1) return DTP_ERR_ARG;
    if (dtype != DTP_BF16) return DTP_ERR_UNSUPPORTED;
    if (!Wqkv_next || !gamma_next || !W_down || !bn || !aligned16(Wqkv_next) || !aligned16(W_down) || !aligned16(bn))
        return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < sq::down_workspace_bytes(H_kv, R, d, N) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemsetAsync(workspace, 0, kWorkspaceHeader, s));
    return sq::launch_down(Wqkv_next, gamma_next, W_down, H_kv, R, d, N, dtype, bn, workspace, s);
}

int dtp_down_finalize(const float* act2, const float* bn, int H_kv, int N, int64_t T_total, float* S_down,
                      void* stream) {
    if (!act2 || !bn || !S_down || H_kv < 1 || H_kv > kMaxHeads || N < 1 || T_total < 1) return DTP_ERR_ARG;
    return launch_down_finalize(act2, bn, H_kv, N, T_total, S_down, static_cast<cudaStream_t>(stream));
}

int dtp_affinity_finalize(float* A, int H_kv, int N, int64_t T_total, const float* wd_sqnorm, void* stream) {
    if (!A || H_kv < 1 || H_kv > kMaxHeads || N < 1 || T_total < 1 || !aligned16(A)) return DTP_ERR_ARG;
    return launch_finalize(A, H_kv, N, T_total, wd_sqnorm, static_cast<cudaStream_t>(stream));
}

int dtp_down_sqnorm(const void* W_down, int d, int N, int dtype, float* out, void* stream) {
    if (!W_down || !out || d < 1 || N < 1 || (dtype != DTP_BF16 && dtype != DTP_F32)) return DTP_ERR_ARG;
    return launch_down_sqnorm(W_down, d, N, dtype, out, static_cast<cudaStream_t>(stream));
}

int dtp_workspace_status(const void* workspace, size_t workspace_bytes, void* stream) {
    if (!workspace || workspace_bytes < kWorkspaceHeader) return DTP_ERR_WORKSPACE;
    int st = 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DTP_CUDA_TRY(cudaMemcpyAsync(&st, workspace, sizeof(int), cudaMemcpyDeviceToHost, s));
    DTP_CUDA_TRY(cudaStreamSynchronize(s));
    return st == 0 ? DTP_OK : st;
}

int dtp_search_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes) {
    if (!bytes || !search_sizes_ok(layers, H_kv, N, D, 1)) return DTP_ERR_ARG;
    *bytes = search::workspace_bytes(layers, H_kv, N, D);
    return DTP_OK;
}

int dtp_search_layout_batched(const float* A, int layers, int H_kv, int N, int D, int iters, int32_t* head_part,
                              int32_t* neuron_dev, int64_t* score_q, double* score, int32_t* iters_done,
                              void* workspace, size_t workspace_bytes, void* stream) {
    if (!search_sizes_ok(layers, H_kv, N, D, iters)) return DTP_ERR_ARG;
    if (!A || !head_part || !neuron_dev || !score_q || !score || !iters_done) return DTP_ERR_ARG;
    if (!aligned16(A)) return DTP_ERR_ARG;
    const size_t need = search::workspace_bytes(layers, H_kv, N, D);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return DTP_ERR_WORKSPACE;
    return search::launch(A, layers, H_kv, N, D, iters, head_part, neuron_dev, score_q, score, iters_done, workspace,
                          static_cast<cudaStream_t>(stream));
}

// The exhaustive search visits at most 2^20 unlabelled partitions per layer.
static bool global_sizes_ok(int layers, int H, int N, int D) {
    return search_sizes_ok(layers, H, N, D, 1) && layers <= 65535 &&
           search::unlabelled_count(H, D) <= (int64_t(1) << 20) &&
           static_cast<int64_t>(layers) * search::unlabelled_count(H, D) <= (int64_t(1) << 26);
}

int dtp_search_global_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes) {
    if (!bytes || !global_sizes_ok(layers, H_kv, N, D)) return DTP_ERR_ARG;
    *bytes = search::global_workspace_bytes(layers, H_kv, N, D);
    return DTP_OK;
}

int dtp_search_global(const float* A, int layers, int H_kv, int N, int D, int32_t* head_part, int32_t* neuron_dev,
                      int64_t* score_q, double* score, void* workspace, size_t workspace_bytes, void* stream) {
    if (!global_sizes_ok(layers, H_kv, N, D)) return DTP_ERR_ARG;
    if (!A || !head_part || !neuron_dev || !score_q || !score || !aligned16(A)) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < search::global_workspace_bytes(layers, H_kv, N, D) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    return search::launch_global(A, layers, H_kv, N, D, head_part, neuron_dev, score_q, score, workspace,
                                 static_cast<cudaStream_t>(stream));
}

int dtp_search_chain_workspace_size(int layers, int H_kv, int N, int D, size_t* bytes) {
    if (!bytes || !search_sizes_ok(layers, H_kv, N, D, 1)) return DTP_ERR_ARG;
    *bytes = search::chain_workspace_bytes(layers, H_kv, N, D);
    return DTP_OK;
}

int dtp_search_chain_ex(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D, int iters,
                        const uint8_t* move_heads, const uint8_t* move_neurons, int minimize, int32_t* head_part,
                        int32_t* neuron_dev, int64_t* J_q, double* J, int32_t* iters_done, void* workspace,
                        size_t workspace_bytes, void* stream) {
    if (!search_sizes_ok(layers, H_kv, N, D, iters)) return DTP_ERR_ARG;
    if (!S_up || (layers > 1 && !S_down) || !head_part || !neuron_dev || !J_q || !J || !iters_done)
        return DTP_ERR_ARG;
    if (!aligned16(S_up) || (S_down && !aligned16(S_down))) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < search::chain_workspace_bytes(layers, H_kv, N, D) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    return search::launch_chain(S_up, S_down, layers, H_kv, N, D, iters, move_heads, move_neurons, minimize,
                                head_part, neuron_dev, J_q, J, iters_done, workspace,
                                static_cast<cudaStream_t>(stream));
}

int dtp_search_chain(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D, int iters,
                     int32_t* head_part, int32_t* neuron_dev, int64_t* J_q, double* J, int32_t* iters_done,
                     void* workspace, size_t workspace_bytes, void* stream) {
    return dtp_search_chain_ex(S_up, S_down, layers, H_kv, N, D, iters, nullptr, nullptr, 0, head_part, neuron_dev,
                               J_q, J, iters_done, workspace, workspace_bytes, stream);
}

int dtp_chain_score(const float* S_up, const float* S_down, int layers, int H_kv, int N, int D,
                    const int32_t* head_part, const int32_t* neuron_dev, int64_t* edge_q, int64_t* J_q, double* J,
                    void* workspace, size_t workspace_bytes, void* stream) {
    if (!search_sizes_ok(layers, H_kv, N, D, 1)) return DTP_ERR_ARG;
    if (!S_up || (layers > 1 && !S_down) || !head_part || !neuron_dev || !J_q || !J) return DTP_ERR_ARG;
    if (!aligned16(S_up) || (S_down && !aligned16(S_down))) return DTP_ERR_ARG;
    if (!workspace || workspace_bytes < search::chain_workspace_bytes(layers, H_kv, N, D) || !aligned16(workspace))
        return DTP_ERR_WORKSPACE;
    return search::launch_chain_score(S_up, S_down, layers, H_kv, N, D, head_part, neuron_dev, edge_q, J_q, J,
                                      workspace, static_cast<cudaStream_t>(stream));
}

int dtp_search_layout(const float* A, int H_kv, int N, int D, int iters, int32_t* head_part, int32_t* neuron_dev,
                      int64_t* score_q, double* score, int32_t* iters_done, void* workspace, size_t workspace_bytes,
                      void* stream) {
    return dtp_search_layout_batched(A, 1, H_kv, N, D, iters, head_part, neuron_dev, score_q, score, iters_done,
                                     workspace, workspace_bytes, stream);
}

}  // extern "C"
