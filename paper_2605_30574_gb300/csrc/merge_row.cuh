// Log-sum-exp merge of one output row.  Warp-cooperative: all 32 lanes of
// the warp must call it.
//
// out = sum_i 2^(m_i - M) o_i / sum_i 2^(m_i - M) l_i over the live partial
// states of the row (M = max m_i), with a ZERO prompt span entering as the
// closed-form state (m = 0, l = #visible prompt positions, o = 0): all-zero
// keys give logit 0 and all-zero values add nothing (Table 1).  A row with no
// live state (nothing visible) outputs 0.
#pragma once

#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"

namespace splice {

__device__ __forceinline__ void merge_row(const AttnParams& P, long row, int lane) {
    const int s = int(row / P.Hq);
    const uint8_t code = P.src[s];
    const int n_pre = code == SPLICE_SRC_ZERO ? 0 : P.nsp;
    const int n = n_pre + P.nss;                       // <= kMaxSplits (16)
    const int p_vis = P.p_hi - P.p_lo;
    const size_t plane = size_t(P.B) * P.Hq;
    // lane i holds partial i's (m, l), so all of them are in flight at once
    const int slot = lane < n_pre ? lane : kMaxPrefixSplits + (lane - n_pre);
    float m = -INFINITY, l = 0.f;
    if (lane < n) {
        const float2 ml = __ldcg(P.ws_ml + size_t(slot) * plane + row);
        m = ml.x;
        l = ml.y;
    }
    const bool zero_span = code == SPLICE_SRC_ZERO && p_vis > 0;
    float M = l > 0.f ? m : -INFINITY;
    if (zero_span) M = fmaxf(M, 0.f);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float w = l > 0.f ? exp2f(m - M) : 0.f;
    float den = w * l;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
    if (zero_span) den += float(p_vis) * exp2f(0.f - M);
    const float inv = den > 0.f ? 1.f / den : 0.f;
    float wall[kMaxSplits];
#pragma unroll
    for (int i = 0; i < kMaxSplits; ++i) wall[i] = __shfl_sync(0xffffffffu, w, i);
    const int c4 = P.D / 4;
    float4* out = reinterpret_cast<float4*>(P.out + size_t(row) * P.D);
    for (int c = lane; c < c4; c += 32) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int i = 0; i < kMaxSplits; ++i) {
            if (i < n && wall[i] != 0.f) {
                const int sl = i < n_pre ? i : kMaxPrefixSplits + (i - n_pre);
                const float4 o = __ldcg(reinterpret_cast<const float4*>(P.ws_o + (size_t(sl) * plane + row) * P.D) + c);
                acc.x = fmaf(wall[i], o.x, acc.x);
                acc.y = fmaf(wall[i], o.y, acc.y);
                acc.z = fmaf(wall[i], o.z, acc.z);
                acc.w = fmaf(wall[i], o.w, acc.w);
            }
        }
        out[c] = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
    }
}

}  // namespace splice
