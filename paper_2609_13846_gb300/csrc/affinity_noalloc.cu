// affinity_noalloc.cu -- dtp_affinity_accumulate_noalloc: the bf16 (tcgen05)
// affinity pass for callers that cannot allocate device memory.
//
// Some callers of this library cannot allocate device memory, nor hand it a
// workspace: a plugin whose host application owns every device allocation
// and exposes none to its plugins, a serving runtime with a fixed memory plan
// that must not grow its device footprint after start-up, or a latency-bound
// loop that may not call cudaMalloc because cudaMalloc can synchronise the
// device.  For them this entry point runs the same kernels as
// dtp_affinity_accumulate with DTP_BF16, but takes its scratch (the status
// word and the per-unit partial sums) from the fixed array below instead of a
// caller workspace.  It calls no allocating routine.
//
// The array lives in device memory of every GPU that loads this library until
// the process exits.  Every call shares it, and the array keeps the last
// call's contents: calls that overlap on the GPU (on different streams, or
// from different host threads without ordering) race on it and must be
// serialised by the caller.  The first call on a device looks up the array's
// device address (cudaGetSymbolAddress) with that device current; make that
// first call before any stream capture begins.  The address is kept for the
// life of the process, so no call may follow a cudaDeviceReset of that device.
//
// Device-side failures (a bounded wait that gave up) are recorded in the
// array's status word, which dtp_affinity_noalloc_status reads back.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "dtp_common.cuh"

namespace dtp {
namespace tc {
size_t workspace_bytes(int64_t T, int d, int G, int N);
int launch(const void* X, const void* C, const void* Wg, const void* Wu, int64_t T, int d, int G, int N, float* A,
           void* workspace, cudaStream_t stream, const float* rms, float* act2);
}  // namespace tc
}  // namespace dtp

// 256-byte status header + 16 MiB of partial sums (512 B per token chunk,
// neuron tile and head): c * ceil(N/128) * H_kv <= 32768 per call, c the
// token-chunk count ceil(T/128) rounded up to an even count (the kernel's CTA
// pairs take chunks two at a time).
static constexpr int64_t kNoAllocMaxUnitHeads = 32768;
static constexpr size_t kNoAllocScratchBytes = dtp::kWorkspaceHeader + (size_t(16) << 20);
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

constexpr int kMaxDevices = 64;
void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mutex;

// Device address of g_noalloc_scratch on the current device.  The symbol's
// name is only a host-side stand-in; its device address is looked up once per
// device, with that device current.
int scratch_address(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DTP_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return DTP_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return DTP_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return DTP_OK;
}

}  // namespace

extern "C" int dtp_affinity_accumulate_noalloc(const void* X, const void* C, const void* W_gate, const void* W_up,
                                               int64_t T, int d, int H_kv, int N, float* A, void* stream) {
    if (T < 0 || d < 8 || (d % 8) != 0 || H_kv < 1 || H_kv > 16 || N < 1) return DTP_ERR_ARG;
    if (T > (int64_t(1) << 31) - 256 || N > (1 << 30)) return DTP_ERR_ARG;
    if (T == 0) return DTP_OK;
    if (!X || !C || !W_gate || !W_up || !A) return DTP_ERR_ARG;
    if (!dtp::aligned16(X) || !dtp::aligned16(C) || !dtp::aligned16(W_gate) || !dtp::aligned16(W_up) ||
        !dtp::aligned16(A))
        return DTP_ERR_ARG;
    const int64_t unit_heads = ((T + 255) / 256) * 2 * ((static_cast<int64_t>(N) + 127) / 128) * H_kv;
    if (unit_heads > kNoAllocMaxUnitHeads || dtp::tc::workspace_bytes(T, d, H_kv, N) > kNoAllocScratchBytes)
        return DTP_ERR_WORKSPACE;
    void* scratch = nullptr;
    const int rc = scratch_address(&scratch);
    if (rc != DTP_OK) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The status word must start at zero; the partial sums are all written before they are read.
    if (cudaMemsetAsync(scratch, 0, dtp::kWorkspaceHeader, s) != cudaSuccess) return DTP_ERR_CUDA;
    return dtp::tc::launch(X, C, W_gate, W_up, T, d, H_kv, N, A, scratch, s, nullptr, nullptr);
}

extern "C" int dtp_affinity_noalloc_status(void* stream) {
    void* scratch = nullptr;
    const int rc = scratch_address(&scratch);
    if (rc != DTP_OK) return rc;
    int st = 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(&st, scratch, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return DTP_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return DTP_ERR_CUDA;
    return st == 0 ? DTP_OK : st;
}
