// A wait that is meant to run out: exercises the bounded-wait and error-word
// path the streaming kernels use, without faulting or hanging the GPU.
#include <cuda_runtime.h>

#include "splice_internal.h"
#include "tc_ptx.cuh"

namespace splice {
namespace {

constexpr unsigned kErrDebugWait = 0x80000000u;

__global__ void wait_timeout_kernel(unsigned* err, unsigned long long limit_ns) {
    __shared__ __align__(8) unsigned long long bar;
    volatile int abort_flag = 0;
    const uint32_t b = tc::smem_u32(&bar);
    tc::mbar_init(b, 1);
    tc::fence_mbar_init();
    // nothing ever arrives: the wait gives up after limit_ns and records it
    tc::mbar_wait(b, 0, &abort_flag, err, kErrDebugWait, limit_ns);
}

}  // namespace

int launch_wait_timeout(unsigned* err, unsigned long long limit_ns, void* stream) {
    wait_timeout_kernel<<<1, 1, 0, static_cast<cudaStream_t>(stream)>>>(err, limit_ns);
    return int(cudaGetLastError());
}

}  // namespace splice
