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

// Partials of one row, in merge order: the prompt-span splits, the
// generated-span splits, then -- a row that reads a delta-encoded donor --
// its delta-row splits.  Those come last so that a delta row whose delta
// rows are empty merges exactly as the same row reading the clean span: its
// extra lanes hold weight 0 where the other row's hold nothing.
struct RowParts {
    int span, suffix, delta;
};

__device__ __forceinline__ RowParts row_parts(const AttnParams& P, uint8_t code) {
    RowParts r{code == SPLICE_SRC_ZERO ? 0 : P.nsp, P.nss, 0};
    if (P.delta_on && code >= SPLICE_SRC_DONOR0 && P.slot_delta[code - SPLICE_SRC_DONOR0]) r.delta = P.nsd;
    return r;
}

// Workspace slot of the row's i-th partial: prompt-span splits at slots
// 0.., delta-row splits right after them, generated-span splits from
// kMaxPrefixSplits on.
__device__ __forceinline__ int merge_slot(int i, const RowParts& r) {
    return i < r.span ? i : (i < r.span + r.suffix ? kMaxPrefixSplits + (i - r.span) : i - r.suffix);
}

// Lane-parallel weights: lane i < n holds partial i's weight 2^(m_i - M);
// returns 1 / (sum of weighted row sums), 0 for a row with nothing live.
__device__ __forceinline__ float merge_weights(const AttnParams& P, int lane, int n, bool zero_span, float2 ml,
                                               float* w_out) {
    const float m = ml.x, l = ml.y;
    float M = (lane < n && l > 0.f) ? m : -INFINITY;
    if (zero_span) M = fmaxf(M, 0.f);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float w = (lane < n && l > 0.f) ? exp2f(m - M) : 0.f;
    float den = w * l;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
    if (zero_span) den = fmaf(float(P.p_hi - P.p_lo), exp2f(0.f - M), den);
    *w_out = w;
    return den > 0.f ? 1.f / den : 0.f;
}

// Rows with at most NF live partials: every load of the row -- lane i's
// (m, l) of partial i and this lane's 16-byte slices of o of every partial --
// is issued before any of them is used, so a row costs one round trip.
template <int D, int NF>
__device__ __forceinline__ bool merge_row_fast(const AttnParams& P, long row, int lane) {
    constexpr int C4 = D / 4;                    // float4 slices of a row
    constexpr int SL = (C4 + 31) / 32;           // slices per lane
    const int s = int(row / P.Hq);
    const uint8_t code = P.src[s];
    const RowParts rp = row_parts(P, code);
    const int n = rp.span + rp.suffix + rp.delta;
    if (n > NF) return false;
    const size_t plane = size_t(P.B) * P.Hq;
    float2 ml = make_float2(-INFINITY, 0.f);
    if (lane < n) ml = __ldcg(P.ws_ml + size_t(merge_slot(lane, rp)) * plane + row);
    float4 ov[NF][SL];
#pragma unroll
    for (int i = 0; i < NF; ++i) {
        const float4* src = reinterpret_cast<const float4*>(P.ws_o + (size_t(merge_slot(i, rp)) * plane + row) * D);
#pragma unroll
        for (int q = 0; q < SL; ++q) {
            const int c = lane + 32 * q;
            ov[i][q] = (i < n && c < C4) ? __ldcg(src + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    float w;
    const float inv = merge_weights(P, lane, n, code == SPLICE_SRC_ZERO && P.p_hi > P.p_lo, ml, &w);
    float4 acc[SL];
#pragma unroll
    for (int q = 0; q < SL; ++q) acc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int i = 0; i < NF; ++i) {
        const float wi = __shfl_sync(0xffffffffu, w, i);
        if (i < n && wi != 0.f) {
#pragma unroll
            for (int q = 0; q < SL; ++q) {
                acc[q].x = fmaf(wi, ov[i][q].x, acc[q].x);
                acc[q].y = fmaf(wi, ov[i][q].y, acc[q].y);
                acc[q].z = fmaf(wi, ov[i][q].z, acc[q].z);
                acc[q].w = fmaf(wi, ov[i][q].w, acc[q].w);
            }
        }
    }
    float4* out = reinterpret_cast<float4*>(P.out + size_t(row) * D);
#pragma unroll
    for (int q = 0; q < SL; ++q) {
        const int c = lane + 32 * q;
        if (c < C4) out[c] = make_float4(acc[q].x * inv, acc[q].y * inv, acc[q].z * inv, acc[q].w * inv);
    }
    return true;
}

// RPW rows per warp (2 or 4), 32 / RPW lanes per row (lanes 0-15 row0,
// 16-31 row0 + 1 for RPW = 2), for rows of at most NF live partials each:
// the loads of all the warp's rows go out at once.  The reductions run over
// the row's lanes with the partials on its first n lanes, so they add the
// same values in the same order as merge_weights over 32 lanes (the other
// lanes hold zeros): the same bits as merge_row_fast.  False (nothing
// written) if any of the rows has more partials.
template <int D, int NF, int RPW>
__device__ __forceinline__ bool merge_rows_group(const AttnParams& P, long row0, int lane) {
    constexpr int LPR = 32 / RPW;                // lanes per row
    static_assert(NF <= LPR, "a row's partials sit on its first lanes");
    constexpr int C4 = D / 4;                    // float4 slices of a row
    constexpr int SL = (C4 + LPR - 1) / LPR;     // slices per lane
    const int half = lane / LPR, hl = lane % LPR;
    const long total = long(P.B) * P.Hq;
    const long row = row0 + half;
    const bool live_row = row < total;
    RowParts rp{0, 0, 0};
    uint8_t code = SPLICE_SRC_CLEAN;
    if (live_row) {
        code = P.src[int(row / P.Hq)];
        rp = row_parts(P, code);
    }
    const int n = rp.span + rp.suffix + rp.delta;
    if (!__all_sync(0xffffffffu, n <= NF)) return false;
    const size_t plane = size_t(total);
    float2 ml = make_float2(-INFINITY, 0.f);
    if (hl < n) ml = __ldcg(P.ws_ml + size_t(merge_slot(hl, rp)) * plane + row);
    float4 ov[NF][SL];
#pragma unroll
    for (int i = 0; i < NF; ++i) {
        const float4* src = reinterpret_cast<const float4*>(P.ws_o + (size_t(merge_slot(i, rp)) * plane + row) * D);
#pragma unroll
        for (int q = 0; q < SL; ++q) {
            const int c = hl + LPR * q;
            ov[i][q] = (i < n && c < C4) ? __ldcg(src + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    // weights over the row's lanes: as merge_weights
    const bool zero_span = code == SPLICE_SRC_ZERO && P.p_hi > P.p_lo;
    float M = (hl < n && ml.y > 0.f) ? ml.x : -INFINITY;
    if (zero_span) M = fmaxf(M, 0.f);
#pragma unroll
    for (int off = LPR / 2; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float w = (hl < n && ml.y > 0.f) ? exp2f(ml.x - M) : 0.f;
    float den = w * ml.y;
#pragma unroll
    for (int off = LPR / 2; off > 0; off >>= 1) den += __shfl_xor_sync(0xffffffffu, den, off);
    if (zero_span) den = fmaf(float(P.p_hi - P.p_lo), exp2f(0.f - M), den);
    const float inv = den > 0.f ? 1.f / den : 0.f;
    float4 acc[SL];
#pragma unroll
    for (int q = 0; q < SL; ++q) acc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int i = 0; i < NF; ++i) {
        const float wi = __shfl_sync(0xffffffffu, w, half * LPR + i);
        if (i < n && wi != 0.f) {
#pragma unroll
            for (int q = 0; q < SL; ++q) {
                acc[q].x = fmaf(wi, ov[i][q].x, acc[q].x);
                acc[q].y = fmaf(wi, ov[i][q].y, acc[q].y);
                acc[q].z = fmaf(wi, ov[i][q].z, acc[q].z);
                acc[q].w = fmaf(wi, ov[i][q].w, acc[q].w);
            }
        }
    }
    if (live_row) {
        float4* out = reinterpret_cast<float4*>(P.out + size_t(row) * D);
#pragma unroll
        for (int q = 0; q < SL; ++q) {
            const int c = hl + LPR * q;
            if (c < C4) out[c] = make_float4(acc[q].x * inv, acc[q].y * inv, acc[q].z * inv, acc[q].w * inv);
        }
    }
    return true;
}

template <int D, int NF>
__device__ __forceinline__ bool merge_rows_fast2(const AttnParams& P, long row0, int lane) {
    return merge_rows_group<D, NF, 2>(P, row0, lane);
}

// Any number of live partials (up to kMaxSplits): weights first, then the o
// slices.
__device__ __forceinline__ void merge_row(const AttnParams& P, long row, int lane) {
    const int s = int(row / P.Hq);
    const uint8_t code = P.src[s];
    const RowParts rp = row_parts(P, code);
    const int n = rp.span + rp.suffix + rp.delta;      // <= kMaxSplits (16)
    const size_t plane = size_t(P.B) * P.Hq;
    float2 ml = make_float2(-INFINITY, 0.f);
    if (lane < n) ml = __ldcg(P.ws_ml + size_t(merge_slot(lane, rp)) * plane + row);
    float w;
    const float inv = merge_weights(P, lane, n, code == SPLICE_SRC_ZERO && P.p_hi > P.p_lo, ml, &w);
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
                const float4 o = __ldcg(reinterpret_cast<const float4*>(
                                            P.ws_o + (size_t(merge_slot(i, rp)) * plane + row) * P.D) + c);
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
