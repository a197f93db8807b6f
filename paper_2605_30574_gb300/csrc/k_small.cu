// Small kernels of the decode step: the generated-span append and the
// log-sum-exp merge of the partial softmax states.
#include <cuda_runtime.h>

#include <cmath>

#include "merge_row.cuh"
#include "splice_internal.h"

namespace splice {
namespace {

// Algorithm 1's forward pass appends the step's generated K/V to the cache:
// entry t-1 of every sequence's generated span, copied bit for bit.
__global__ void append_kernel(const uint4* __restrict__ kn, const uint4* __restrict__ vn,
                              uint4* __restrict__ ks, uint4* __restrict__ vs, int B, int N,
                              int Hkv, int chunks, int T, int layer, int slot) {
    // the attention call that usually follows may start launching now (it
    // waits for this grid before it reads anything)
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const long i = long(blockIdx.x) * blockDim.x + threadIdx.x;
    const long total = long(B) * Hkv * chunks;
    if (i >= total) return;
    const int c = int(i % chunks);
    const long sh = i / chunks;          // s * Hkv + h
    const int h = int(sh % Hkv);
    const long s = sh / Hkv;
    const size_t dst = (((size_t(s) * N + layer) * Hkv + h) * size_t(T) + slot) * chunks + c;
    ks[dst] = kn[i];
    vs[dst] = vn[i];
}

// The partial states of the prompt-span and the generated-span passes (and
// the ZERO closed form) -> out.  Rows with up to four partials -- the common
// case -- take a one-round-trip path: for d <= 128 a warp merges two rows,
// one per half-warp; for d = 256 one row per warp.  Rows with more partials
// take the general path, a warp per row.
template <int D>
__global__ void __launch_bounds__(256, 5) merge_kernel(AttnParams P) {
    // Launched behind the prompt-span pass as a programmatic dependent, this
    // grid may start before that pass has finished: wait for it (and so for
    // the generated-span pass it waited for) before reading any partial.
    // A no-op for a plain launch.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long warp = (long(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const long total = long(P.B) * P.Hq;
    if constexpr (D <= 128) {
        const long row0 = 2 * warp;
        if (row0 >= total) return;
        if (merge_rows_fast2<D, 4>(P, row0, lane)) return;
        merge_row(P, row0, lane);
        if (row0 + 1 < total) merge_row(P, row0 + 1, lane);
    } else {
        if (warp >= total) return;
        if (!merge_row_fast<D, 4>(P, warp, lane)) merge_row(P, warp, lane);
    }
}

// Calls whose rows have at most two partials each (one prompt-span split and
// one generated-span split, or fewer): four rows per warp, a quarter-warp per
// row, so twice the rows per warp are in flight; the same bits as the
// two-row path.
template <int D>
__global__ void __launch_bounds__(256, 3) merge_kernel4(AttnParams P) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long warp = (long(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const long total = long(P.B) * P.Hq;
    const long row0 = 4 * warp;
    if (row0 >= total) return;
    if (merge_rows_group<D, 2, 4>(P, row0, lane)) return;
    for (long r = row0; r < row0 + 4 && r < total; r += 2)
        if (!merge_rows_fast2<D, 4>(P, r, lane)) {
            merge_row(P, r, lane);
            if (r + 1 < total) merge_row(P, r + 1, lane);
        }
}

}  // namespace

int launch_append(const uint16_t* kn, const uint16_t* vn, uint16_t* ks, uint16_t* vs, int B, int N,
                  int Hkv, int D, int T, int layer, int step, void* stream) {
    const int chunks = D / 8;
    const long total = long(B) * Hkv * chunks;
    const int block = 256;
    append_kernel<<<unsigned((total + block - 1) / block), block, 0, static_cast<cudaStream_t>(stream)>>>(
        reinterpret_cast<const uint4*>(kn), reinterpret_cast<const uint4*>(vn),
        reinterpret_cast<uint4*>(ks), reinterpret_cast<uint4*>(vs), B, N, Hkv, chunks, T, layer,
        step - 1);
    return int(cudaGetLastError());
}

int launch_merge(const AttnParams& p, void* stream, bool overlap_previous) {
    const long rows = long(p.B) * p.Hq;
    const int block = 256;
    // at most two partials per row: the prompt-span splits (none for a ZERO
    // row), the generated-span splits and a delta row's splits
    const bool four = p.D <= 128 && p.nsp + p.nss + (p.delta_on ? p.nsd : 0) <= 2;
    const long warps = four ? (rows + 3) / 4 : (p.D <= 128 ? (rows + 1) / 2 : rows);
    const long threads = warps * 32;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned((threads + block - 1) / block));
    cfg.blockDim = dim3(block);
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = overlap_previous ? 1 : 0;
    if (four) {
        if (p.D == 64) return int(cudaLaunchKernelEx(&cfg, merge_kernel4<64>, p));
        return int(cudaLaunchKernelEx(&cfg, merge_kernel4<128>, p));
    }
    switch (p.D) {
        case 64: return int(cudaLaunchKernelEx(&cfg, merge_kernel<64>, p));
        case 128: return int(cudaLaunchKernelEx(&cfg, merge_kernel<128>, p));
        case 256: return int(cudaLaunchKernelEx(&cfg, merge_kernel<256>, p));
        default: return int(cudaErrorInvalidValue);
    }
}

}  // namespace splice
