// Test kernels.  A wait that is meant to run out: exercises the bounded-wait
// and error-word path the streaming kernels use, without faulting or hanging
// the GPU.  A late copy: a producer that lets its programmatic dependents
// launch at once but writes its output only after a delay, so a consumer
// that reads before its own griddepcontrol.wait would see stale data.
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

// Lets dependents launch, spins for delay_ns of wall time (bounded by the
// clock, not by any other agent), then copies n16 16-byte words.
__global__ void late_copy_kernel(uint4* __restrict__ dst, const uint4* __restrict__ src, long n16,
                                 unsigned long long delay_ns) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const unsigned long long t0 = tc::globaltimer_ns();
    while (tc::globaltimer_ns() - t0 < delay_ns) __nanosleep(1000);
    for (long i = long(blockIdx.x) * blockDim.x + threadIdx.x; i < n16; i += long(gridDim.x) * blockDim.x)
        dst[i] = src[i];
}

}  // namespace

int launch_late_copy(void* dst, const void* src, size_t bytes, unsigned long long delay_ns, void* stream) {
    const long n16 = long(bytes / 16);
    late_copy_kernel<<<8, 256, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<uint4*>(dst),
                                                                      static_cast<const uint4*>(src), n16, delay_ns);
    return int(cudaGetLastError());
}

int launch_wait_timeout(unsigned* err, unsigned long long limit_ns, void* stream) {
    wait_timeout_kernel<<<1, 1, 0, static_cast<cudaStream_t>(stream)>>>(err, limit_ns);
    return int(cudaGetLastError());
}

}  // namespace splice
