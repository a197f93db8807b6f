// Delta encoding of the stored donor spans against the clean spans.
//
// A stored donor span (prompt p, stored slot st, layer l, kv head h) is
// aligned position by position with the clean span of (p, l, h): §3 trims
// donor and target prompts to the same length.  Position j is encoded iff
// the donor's K row or V row at j differs bit for bit from the clean span's.
// Attention over the donor span is then the log-sum-exp merge of attention
// over the clean span without the encoded positions and attention over the
// encoded rows, so readers of a donor that shares most positions with the
// clean prompt read the clean span (which its clean readers read anyway)
// plus a short run of encoded rows.
//
// One CTA per span:
//   1. each warp compares whole rows of its positions (16-byte chunks, K then
//      V) and sets the position's bit in a shared bitmask;
//   2. a block-wide scan of the words' population counts gives every word's
//      first output row and the span's count;
//   3. the donor rows of the encoded positions are copied in position order
//      to rows 0 .. count-1 of the span's rows in the delta store, and rows
//      count .. T_p-1 are zeroed, so a 128-row tile that runs past the count
//      reads zeros, never stale memory.
#include <cuda_runtime.h>

#include "splice_internal.h"

namespace splice {
namespace {

constexpr int kDeltaThreads = 256;

__global__ void __launch_bounds__(kDeltaThreads) delta_build_kernel(
    const uint4* __restrict__ kc, const uint4* __restrict__ vc, const uint4* __restrict__ kd,
    const uint4* __restrict__ vd, uint32_t* __restrict__ mask, int32_t* __restrict__ count, uint4* __restrict__ xk,
    uint4* __restrict__ xv, int Dst, int N, int Hkv, int Tp, int C, int w32) {
    extern __shared__ uint32_t sm[];                   // [w32] position bits, [w32] first row of each word
    __shared__ int warp_sum[kDeltaThreads / 32];
    uint32_t* bits = sm;
    int* first = reinterpret_cast<int*>(sm + w32);
    const long sp = blockIdx.x;                        // ((p * Dst + st) * N + l) * Hkv + h
    const long h = sp % Hkv;
    const long l = (sp / Hkv) % N;
    const long p = sp / (long(Hkv) * N * Dst);
    const size_t crow = size_t((p * N + l) * Hkv + h) * size_t(Tp);   // first row of the clean span
    const size_t drow = size_t(sp) * size_t(Tp);                      // of the donor span and of its delta rows
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;

    for (int i = threadIdx.x; i < w32; i += blockDim.x) bits[i] = 0u;
    __syncthreads();
    // 1. positions whose K or V row differs
    for (int j = warp; j < Tp; j += nw) {
        bool diff = false;
        for (int c = lane; c < 2 * C; c += 32) {
            const bool is_k = c < C;
            const int cc = is_k ? c : c - C;
            const uint4 a = is_k ? kc[(crow + j) * C + cc] : vc[(crow + j) * C + cc];
            const uint4 b = is_k ? kd[(drow + j) * C + cc] : vd[(drow + j) * C + cc];
            diff |= (a.x != b.x) | (a.y != b.y) | (a.z != b.z) | (a.w != b.w);
        }
        if (__any_sync(0xffffffffu, diff) && lane == 0) atomicOr(&bits[j >> 5], 1u << (j & 31));
    }
    __syncthreads();
    // 2. exclusive scan of the words' population counts (each thread owns a
    //    contiguous run of words)
    const int per = (w32 + int(blockDim.x) - 1) / int(blockDim.x);
    const int w0 = min(w32, int(threadIdx.x) * per), w1 = min(w32, w0 + per);
    int mine = 0;
    for (int w = w0; w < w1; ++w) mine += __popc(bits[w]);
    int incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += v;
    }
    if (lane == 31) warp_sum[warp] = incl;
    __syncthreads();
    int base = 0, total = 0;
    for (int w = 0; w < nw; ++w) {
        if (w < warp) base += warp_sum[w];
        total += warp_sum[w];
    }
    int run = base + incl - mine;
    for (int w = w0; w < w1; ++w) {
        first[w] = run;
        run += __popc(bits[w]);
    }
    __syncthreads();
    // 3. encoded rows in position order, then zeros
    for (int j = warp; j < Tp; j += nw) {
        const uint32_t word = bits[j >> 5];
        if (!((word >> (j & 31)) & 1u)) continue;
        const size_t r = size_t(first[j >> 5] + __popc(word & ((1u << (j & 31)) - 1u)));
        for (int c = lane; c < C; c += 32) {
            xk[(drow + r) * C + c] = kd[(drow + j) * C + c];
            xv[(drow + r) * C + c] = vd[(drow + j) * C + c];
        }
    }
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    for (size_t i = size_t(total) * C + threadIdx.x; i < size_t(Tp) * C; i += blockDim.x) {
        xk[drow * C + i] = z;
        xv[drow * C + i] = z;
    }
    for (int i = threadIdx.x; i < w32; i += blockDim.x) mask[size_t(sp) * w32 + i] = bits[i];
    if (threadIdx.x == 0) count[sp] = total;
}

}  // namespace

int launch_delta_build(const uint16_t* kc, const uint16_t* vc, const uint16_t* kd, const uint16_t* vd,
                       uint32_t* mask, int32_t* count, uint16_t* xk, uint16_t* xv, int P, int Dst, int N,
                       int Hkv, int Tp, int D, int w32, void* stream) {
    const long spans = long(P) * Dst * N * Hkv;
    if (spans <= 0) return 0;
    const size_t smem = size_t(w32) * 8;
    if (smem > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(delta_build_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             int(smem));
        if (e != cudaSuccess) return int(e);
    }
    delta_build_kernel<<<unsigned(spans), kDeltaThreads, smem, static_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<const uint4*>(kc), reinterpret_cast<const uint4*>(vc), reinterpret_cast<const uint4*>(kd),
        reinterpret_cast<const uint4*>(vd), mask, count, reinterpret_cast<uint4*>(xk), reinterpret_cast<uint4*>(xv),
        Dst, N, Hkv, Tp, D / 8, w32);
    return int(cudaGetLastError());
}

}  // namespace splice
