// spliced_decode_attn_static: the decode-attention entry point for callers
// that cannot allocate device memory (see include/splice.h).
//
// The partial softmax states that spliced_decode_attn keeps in a caller-
// provided workspace live here in a fixed-size file-scope device array
// instead.  This file only locates that array on the calling device and hands
// it to the regular entry point; it allocates nothing.
#include <cuda_runtime.h>

#include <cstdio>
#include <mutex>

#include "splice_internal.h"

namespace {

// Scratch shared by every call on a device.  Every GPU that loads this
// library holds SPLICE_STATIC_SCRATCH_BYTES of device memory for it until the
// process exits.
__device__ __align__(256) unsigned char g_static_scratch[SPLICE_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on `device`, found once per device
// with that device current.  The host-side name g_static_scratch is only a
// stand-in for the symbol and must never be passed to a kernel.
cudaError_t scratch_on(int device, void** out) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_scratch_ptr[device]) {
        *out = g_scratch_ptr[device];
        return cudaSuccess;
    }
    int prev = -1;
    cudaError_t e = cudaGetDevice(&prev);
    if (e != cudaSuccess) return e;
    if (prev != device && (e = cudaSetDevice(device)) != cudaSuccess) return e;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (prev != device) cudaSetDevice(prev);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[device] = p;
    *out = p;
    return cudaSuccess;
}

}  // namespace

extern "C" {

splice_status spliced_decode_attn_static(splice_desc* desc, int layer, int step, const splice_bf16* q,
                                         const splice_bf16* k_clean, const splice_bf16* v_clean,
                                         const splice_bf16* k_donor, const splice_bf16* v_donor,
                                         const splice_bf16* k_suffix, const splice_bf16* v_suffix,
                                         float* out, void* stream) {
    if (!desc || !q) return spliced_decode_attn(desc, layer, step, q, k_clean, v_clean, k_donor, v_donor,
                                                k_suffix, v_suffix, out, nullptr, 0, stream);
    const size_t need = splice_workspace_bytes(desc);
    if (need > SPLICE_STATIC_SCRATCH_BYTES) {
        char msg[256];
        std::snprintf(msg, sizeof msg,
                      "spliced_decode_attn_static: this descriptor needs %zu bytes of scratch, more than the "
                      "static maximum of %zu bytes; use spliced_decode_attn with a workspace",
                      need, size_t(SPLICE_STATIC_SCRATCH_BYTES));
        splice::set_last_error(msg);
        return SPLICE_EINVAL;
    }
    // The scratch lives on the device that holds the tensors.
    cudaPointerAttributes attr{};
    cudaError_t e = cudaPointerGetAttributes(&attr, q);
    if (e != cudaSuccess || attr.type != cudaMemoryTypeDevice || attr.device < 0 || attr.device >= kMaxDevices) {
        cudaGetLastError();
        splice::set_last_error("spliced_decode_attn_static: q is not a device pointer");
        return SPLICE_EINVAL;
    }
    void* scratch = nullptr;
    e = scratch_on(attr.device, &scratch);
    if (e != cudaSuccess) {
        char msg[256];
        std::snprintf(msg, sizeof msg, "spliced_decode_attn_static: cudaGetSymbolAddress failed: %s",
                      cudaGetErrorString(e));
        splice::set_last_error(msg);
        return SPLICE_ECUDA;
    }
    return spliced_decode_attn(desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                               out, scratch, SPLICE_STATIC_SCRATCH_BYTES, stream);
}

}  // extern "C"
