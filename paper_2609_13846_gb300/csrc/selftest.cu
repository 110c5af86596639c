// selftest.cu -- dtp_selftest_bounded_wait: exercises, on the GPU, the bounded
// mbarrier wait every kernel of this library uses, so that a caller (or a test)
// can check that a device-side wait which is never satisfied gives up and
// reports through the workspace status word instead of hanging, and that the
// other waits of the block follow it out through the shared abort flag.
#include <cuda_runtime.h>
#include <stdint.h>

#include "dtp_common.cuh"

namespace {

// Thread 0 waits on barrier a with the caller's limit; thread 64 waits on
// barrier b (never completed) with the library's full limit and must leave as
// soon as thread 0 gives up.  With `complete`, thread 32 arrives on a first.
__global__ void selftest_wait_kernel(int* status, unsigned long long* elapsed, uint64_t limit_ns, int complete) {
    __shared__ uint64_t bar_a, bar_b;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        dtp::mbar_init(dtp::smem_u32(&bar_a), 1);
        dtp::mbar_init(dtp::smem_u32(&bar_b), 1);
        abort_flag = 0;
        dtp::fence_mbar_init();
    }
    __syncthreads();
    volatile int* abort = &abort_flag;
    if (threadIdx.x == 32 && complete) dtp::mbar_arrive(dtp::smem_u32(&bar_a));
    if (threadIdx.x == 0) {
        const uint64_t t0 = dtp::globaltimer_ns();
        const bool ok = dtp::mbar_wait(dtp::smem_u32(&bar_a), 0, abort, limit_ns);
        elapsed[0] = dtp::globaltimer_ns() - t0;
        if (!ok) atomicExch(status, static_cast<int>(DTP_ERR_NOT_CONVERGED));
    }
    if (threadIdx.x == 64 && !complete) {
        const uint64_t t0 = dtp::globaltimer_ns();
        dtp::mbar_wait(dtp::smem_u32(&bar_b), 0, abort);
        elapsed[1] = dtp::globaltimer_ns() - t0;
    }
}

}  // namespace

extern "C" int dtp_selftest_bounded_wait(uint64_t limit_ns, int complete, void* workspace, size_t workspace_bytes,
                                         uint64_t* elapsed_ns, void* stream) {
    if (!workspace || workspace_bytes < dtp::kWorkspaceHeader || !elapsed_ns) return DTP_ERR_ARG;
    if (limit_ns < 1000 || limit_ns > 1000000000ull || (complete != 0 && complete != 1)) return DTP_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    unsigned long long* elapsed = reinterpret_cast<unsigned long long*>(ws + 64);
    DTP_CUDA_TRY(cudaMemsetAsync(ws, 0, dtp::kWorkspaceHeader, s));
    selftest_wait_kernel<<<1, 96, 0, s>>>(reinterpret_cast<int*>(ws), elapsed, limit_ns, complete);
    DTP_CUDA_TRY(cudaGetLastError());
    unsigned long long host[2] = {0, 0};
    DTP_CUDA_TRY(cudaMemcpyAsync(host, elapsed, sizeof(host), cudaMemcpyDeviceToHost, s));
    DTP_CUDA_TRY(cudaStreamSynchronize(s));
    elapsed_ns[0] = host[0];
    elapsed_ns[1] = host[1];
    return DTP_OK;
}
