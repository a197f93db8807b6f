// spliced_decode_attn_static: the decode-attention entry point for callers
// that cannot allocate device memory (see include/splice.h).
//
// The partial softmax states that spliced_decode_attn keeps in a caller-
// provided workspace live here in a fixed-size file-scope device array
// instead.  This file only locates that array on the descriptor's device and
// hands it to the regular entry point; it allocates nothing.
#include <cuda.h>
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
unsigned long long g_scratch_ctx[kMaxDevices] = {};   // context the address belongs to

// cuCtxGetCurrent and cuCtxGetId through the runtime's driver entry point
// (no -lcuda): a device reset gives the device a new primary context, and
// with it a new address for the array.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

unsigned long long current_context_id() {
    static CtxGetCurrentFn get_cur = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static bool looked = false;
    if (!looked) {
        looked = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_cur = reinterpret_cast<CtxGetCurrentFn>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<CtxGetIdFn>(p);
    }
    CUcontext c = nullptr;
    unsigned long long id = 0;
    if (!get_cur || !get_id || get_cur(&c) != CUDA_SUCCESS || !c || get_id(c, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array on `device`, which must be current.
// Looked up once per device, and again if the device's context changed
// since (after a cudaDeviceReset).  The host-side name g_static_scratch is
// only a stand-in for the symbol and must never be passed to a kernel.
cudaError_t scratch_on(int device, void** out) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    unsigned long long ctx = current_context_id();   // 0: no context bound to this thread yet
    if (g_scratch_ptr[device] && ctx != 0 && ctx == g_scratch_ctx[device]) {
        *out = g_scratch_ptr[device];
        return cudaSuccess;
    }
    void* p = nullptr;
    // (binds the device's primary context to this thread if it was not)
    cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    if (ctx == 0) ctx = current_context_id();
    g_scratch_ptr[device] = p;
    g_scratch_ctx[device] = ctx;
    *out = p;
    return cudaSuccess;
}

}  // namespace

extern "C" {

size_t splice_static_scratch_bytes(void) { return size_t(SPLICE_STATIC_SCRATCH_BYTES); }

splice_status spliced_decode_attn_static(splice_desc* desc, int layer, int step, const splice_bf16* q,
                                         const splice_bf16* k_clean, const splice_bf16* v_clean,
                                         const splice_bf16* k_donor, const splice_bf16* v_donor,
                                         const splice_bf16* k_suffix, const splice_bf16* v_suffix,
                                         float* out, void* stream) {
    if (!desc)   // the regular entry point reports it
        return spliced_decode_attn(desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                                   out, nullptr, 0, stream);
    // the size limit first: it holds whatever the other arguments are
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
    const int device = splice::desc_device(desc);
    if (device < 0 || !q)   // host-only descriptor, NULL q: the regular entry point reports these
        return spliced_decode_attn(desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                                   out, nullptr, 0, stream);
    if (device >= kMaxDevices) {
        splice::set_last_error("spliced_decode_attn_static: device ordinal beyond the library's table");
        return SPLICE_EINVAL;
    }
    // The kernels run on the descriptor's device, so the scratch must be
    // that device's array; a q on another device would make them read a
    // peer's memory.  (Managed memory is accepted, as by the regular entry
    // point.)
    cudaPointerAttributes attr{};
    cudaError_t e = cudaPointerGetAttributes(&attr, q);
    if (e != cudaSuccess) {
        cudaGetLastError();
        splice::set_last_error("spliced_decode_attn_static: q is not a CUDA pointer");
        return SPLICE_EINVAL;
    }
    if (attr.type == cudaMemoryTypeDevice && attr.device != device) {
        char msg[160];
        std::snprintf(msg, sizeof msg, "spliced_decode_attn_static: q is on device %d, the descriptor on device %d",
                      attr.device, device);
        splice::set_last_error(msg);
        return SPLICE_EINVAL;
    }
    if (attr.type != cudaMemoryTypeDevice && attr.type != cudaMemoryTypeManaged) {
        splice::set_last_error("spliced_decode_attn_static: q is not device or managed memory");
        return SPLICE_EINVAL;
    }
    int prev = -1;
    e = cudaGetDevice(&prev);
    if (e == cudaSuccess && prev != device) e = cudaSetDevice(device);
    void* scratch = nullptr;
    if (e == cudaSuccess) e = scratch_on(device, &scratch);
    if (prev >= 0 && prev != device) cudaSetDevice(prev);
    if (e != cudaSuccess) {
        char msg[256];
        std::snprintf(msg, sizeof msg, "spliced_decode_attn_static: locating the static scratch failed: %s",
                      cudaGetErrorString(e));
        splice::set_last_error(msg);
        return SPLICE_ECUDA;
    }
    return spliced_decode_attn(desc, layer, step, q, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                               out, scratch, SPLICE_STATIC_SCRATCH_BYTES, stream);
}

}  // extern "C"
