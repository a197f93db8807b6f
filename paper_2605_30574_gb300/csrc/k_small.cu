// Small kernels of the decode step: the generated-span append and the
// log-sum-exp merge of the partial softmax states.
#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"

namespace splice {
namespace {

// Algorithm 1's forward pass appends the step's generated K/V to the cache:
// entry t-1 of every sequence's generated span, copied bit for bit.
__global__ void append_kernel(const uint4* __restrict__ kn, const uint4* __restrict__ vn,
                              uint4* __restrict__ ks, uint4* __restrict__ vs, int B, int N,
                              int Hkv, int chunks, int T, int layer, int slot) {
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

// out = sum_i 2^(m_i - M) o_i / sum_i 2^(m_i - M) l_i over the live partial
// states of a row (M = max m_i), with a ZERO prompt span entering as the
// closed-form state (m = 0, l = #visible prompt positions, o = 0): all-zero
// keys give logit 0 and all-zero values add nothing (Table 1).
__global__ void merge_kernel(AttnParams P) {
    const long warp = (long(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    const long rows = long(P.B) * P.Hq;
    if (warp >= rows) return;
    const int s = int(warp / P.Hq);
    const uint8_t code = P.src[s];
    const int n_pre = code == SPLICE_SRC_ZERO ? 0 : P.nsp;
    const int p_vis = P.p_hi - P.p_lo;
    const size_t plane = size_t(P.B) * P.Hq;

    float ms[kMaxSplits], ls[kMaxSplits];
    int slots[kMaxSplits];
    int n = 0;
    float M = -INFINITY;
    for (int i = 0; i < n_pre; ++i) {
        const float2 ml = P.ws_ml[size_t(i) * plane + warp];
        slots[n] = i;
        ms[n] = ml.x;
        ls[n] = ml.y;
        if (ml.y > 0.f) M = fmaxf(M, ml.x);
        ++n;
    }
    for (int i = 0; i < P.nss; ++i) {
        const int sl = kMaxPrefixSplits + i;
        const float2 ml = P.ws_ml[size_t(sl) * plane + warp];
        slots[n] = sl;
        ms[n] = ml.x;
        ls[n] = ml.y;
        if (ml.y > 0.f) M = fmaxf(M, ml.x);
        ++n;
    }
    const bool zero_span = code == SPLICE_SRC_ZERO && p_vis > 0;
    if (zero_span) M = fmaxf(M, 0.f);

    float den = zero_span ? float(p_vis) * exp2f(0.f - M) : 0.f;
    float w[kMaxSplits];
    for (int i = 0; i < n; ++i) {
        w[i] = ls[i] > 0.f ? exp2f(ms[i] - M) : 0.f;
        den += w[i] * ls[i];
    }
    const float inv = den > 0.f ? 1.f / den : 0.f;
    const int c4 = P.D / 4;
    float4* out = reinterpret_cast<float4*>(P.out + size_t(warp) * P.D);
    for (int c = lane; c < c4; c += 32) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int i = 0; i < n; ++i) {
            if (w[i] == 0.f) continue;
            const float4 o = reinterpret_cast<const float4*>(
                P.ws_o + (size_t(slots[i]) * plane + warp) * P.D)[c];
            acc.x = fmaf(w[i], o.x, acc.x);
            acc.y = fmaf(w[i], o.y, acc.y);
            acc.z = fmaf(w[i], o.z, acc.z);
            acc.w = fmaf(w[i], o.w, acc.w);
        }
        out[c] = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
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

int launch_merge(const AttnParams& p, void* stream) {
    const long rows = long(p.B) * p.Hq;
    const int block = 256;
    const long threads = rows * 32;
    merge_kernel<<<unsigned((threads + block - 1) / block), block, 0, static_cast<cudaStream_t>(stream)>>>(p);
    return int(cudaGetLastError());
}

}  // namespace splice
