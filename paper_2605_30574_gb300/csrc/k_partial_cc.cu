// CUDA-core attention partials: for one (sequence s, kv head h, key split)
// a warp streams a contiguous run of keys of one K/V block and emits, for each
// of the G query rows of that kv head, the partial softmax state
// (m, l, o[d]): m = running reference max of the logits (log2 units),
// l = sum 2^(z - m), o = sum 2^(z - m) v.  The merge kernel combines the
// partials of the prompt span and of the generated span (§3: a decode step
// attends over both).
//
// Lane mapping: a key row of d bf16 is split over LPK = d / 16 lanes, each
// holding 16 dims as two 16-byte chunks (chunk c and c + LPK, so every load
// instruction reads whole 16-byte runs of consecutive lanes); a warp works
// on KPW = 32 / LPK keys at once, U keys per lane group per iteration.  The
// U * G partial dot products of a lane are summed across its LPK lanes with a
// butterfly reduce-scatter + all-gather (fewer shuffles than one all-reduce
// per value).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"

namespace splice {
namespace {

constexpr unsigned kFull = 0xffffffffu;
// Lazy-rescale threshold (log2 units): the reference max only moves when a
// block's max exceeds it by more than this, so p = 2^(z - m) <= 2^8.
constexpr float kTau = 8.0f;

__host__ __device__ constexpr int ilog2(int x) { return x <= 1 ? 0 : 1 + ilog2(x / 2); }

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

// Sum NV values over the LPK lanes of a lane group (xor offsets < LPK);
// every lane ends with all NV sums.
template <int NV, int LPK>
__device__ __forceinline__ void group_allreduce(float (&v)[NV], int lane) {
    constexpr int LOG_LPK = ilog2(LPK);
    constexpr int LOG_NV = ilog2(NV);
    constexpr int SPLITS = LOG_NV < LOG_LPK ? LOG_NV : LOG_LPK;
#pragma unroll
    for (int lv = 0; lv < LOG_LPK; ++lv) {
        const int o = LPK >> (lv + 1);
        const bool up = (lane & o) != 0;
        if (lv < SPLITS) {
            const int h = NV >> (lv + 1);
#pragma unroll
            for (int i = 0; i < h; ++i) {
                const float send = up ? v[i] : v[i + h];
                const float keep = up ? v[i + h] : v[i];
                v[i] = keep + __shfl_xor_sync(kFull, send, o);
            }
        } else {
            v[0] += __shfl_xor_sync(kFull, v[0], o);
        }
    }
#pragma unroll
    for (int lv = SPLITS - 1; lv >= 0; --lv) {
        const int o = LPK >> (lv + 1);
        const bool up = (lane & o) != 0;
        const int h = NV >> (lv + 1);
        float r[NV / 2 > 0 ? NV / 2 : 1];
#pragma unroll
        for (int i = 0; i < h; ++i) r[i] = __shfl_xor_sync(kFull, v[i], o);
#pragma unroll
        for (int i = 0; i < h; ++i) {
            const float mine = v[i];
            v[i] = up ? r[i] : mine;
            v[i + h] = up ? mine : r[i];
        }
    }
}

template <int D, int GT>
struct CC {
    static constexpr int DPL = 16;
    static constexpr int LPK = D / DPL;
    static constexpr int KPW = 32 / LPK;
    static constexpr int U = 2;
    static constexpr int NV = U * GT;
};

// One warp per work item.  Items: (s, h, row chunk rc, split).  prefix=true
// reads the sequence's prompt-span source; otherwise its generated span.
template <int D, int GT>
__global__ void __launch_bounds__(128) partials_cc_kernel(AttnParams P, int prefix, int n_items) {
    using C = CC<D, GT>;
    const int lane = threadIdx.x & 31;
    const int item = blockIdx.x * 4 + (threadIdx.x >> 5);
    if (item >= n_items) return;
    const int nsplit = prefix ? P.nsp : P.nss;
    const int n_rc = P.G / GT;
    int rem = item;
    const int split = rem % nsplit;
    rem /= nsplit;
    const int rc = rem % n_rc;
    rem /= n_rc;
    const int h = rem % P.Hkv;
    const int s = rem / P.Hkv;

    const uint16_t* kb;
    const uint16_t* vb;
    int k0, k1;
    if (prefix) {
        const uint8_t code = P.src[s];
        if (code == SPLICE_SRC_ZERO) return;   // closed form, folded in by the merge
        const int p = P.seq_prompt[s];
        size_t span;
        if (code == SPLICE_SRC_CLEAN) {
            span = (size_t(p) * P.N + P.layer) * P.Hkv + h;
            kb = P.kc;
            vb = P.vc;
        } else {
            const int st = P.slot_stored[code - SPLICE_SRC_DONOR0];
            span = ((size_t(p) * P.Dst + st) * P.N + P.layer) * P.Hkv + h;
            kb = P.kd;
            vb = P.vd;
        }
        kb += span * P.Tp * D;
        vb += span * P.Tp * D;
        k0 = P.p_lo + split * P.p_chunk;
        k1 = min(P.p_hi, k0 + P.p_chunk);
    } else {
        const size_t blk = ((size_t(s) * P.N + P.layer) * P.Hkv + h) * size_t(P.T);
        kb = P.ks + blk * D;
        vb = P.vs + blk * D;
        k0 = P.s_lo + split * P.s_chunk;
        k1 = min(P.s_hi, k0 + P.s_chunk);
    }

    const int gi = lane / C::LPK;   // lane group: which key of a KPW-wide step
    const int dl = lane % C::LPK;   // which 16-dim slice
    const int c0 = dl, c1 = dl + C::LPK;   // 16-byte chunks held by this lane

    // q rows pre-scaled into log2 units.
    float q[GT][16];
#pragma unroll
    for (int g = 0; g < GT; ++g) {
        const int hq = h * P.G + rc * GT + g;
        const uint4* qr = reinterpret_cast<const uint4*>(P.q + (size_t(s) * P.Hq + hq) * D);
        float a[8], b[8];
        bf16x8_to_f32(qr[c0], a);
        bf16x8_to_f32(qr[c1], b);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            q[g][i] = a[i] * P.scale_log2;
            q[g][8 + i] = b[i] * P.scale_log2;
        }
    }

    float m[GT], l[GT], o[GT][16];
#pragma unroll
    for (int g = 0; g < GT; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
#pragma unroll
        for (int i = 0; i < 16; ++i) o[g][i] = 0.f;
    }

    for (int base = k0; base < k1; base += C::U * C::KPW) {
        uint4 kr[C::U][2], vr[C::U][2];
        bool valid[C::U];
#pragma unroll
        for (int u = 0; u < C::U; ++u) {
            const int j = base + u * C::KPW + gi;
            valid[u] = j < k1;
            const int jj = valid[u] ? j : k0;
            const uint4* kp = reinterpret_cast<const uint4*>(kb + size_t(jj) * D);
            const uint4* vp = reinterpret_cast<const uint4*>(vb + size_t(jj) * D);
            kr[u][0] = __ldg(kp + c0);
            kr[u][1] = __ldg(kp + c1);
            vr[u][0] = __ldg(vp + c0);
            vr[u][1] = __ldg(vp + c1);
        }
        float sc[C::NV];
#pragma unroll
        for (int u = 0; u < C::U; ++u) {
            float ka[8], kb8[8];
            bf16x8_to_f32(kr[u][0], ka);
            bf16x8_to_f32(kr[u][1], kb8);
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                float acc = 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) acc = fmaf(q[g][i], ka[i], acc);
#pragma unroll
                for (int i = 0; i < 8; ++i) acc = fmaf(q[g][8 + i], kb8[i], acc);
                sc[u * GT + g] = acc;
            }
        }
        group_allreduce<C::NV, C::LPK>(sc, lane);
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            float mb = -INFINITY;
#pragma unroll
            for (int u = 0; u < C::U; ++u)
                if (valid[u]) mb = fmaxf(mb, sc[u * GT + g]);
            if (mb > m[g] + kTau) {
                const float alpha = exp2f(m[g] - mb);
                l[g] *= alpha;
#pragma unroll
                for (int i = 0; i < 16; ++i) o[g][i] *= alpha;
                m[g] = mb;
            }
        }
#pragma unroll
        for (int u = 0; u < C::U; ++u) {
            float va[8], vb8[8];
            bf16x8_to_f32(vr[u][0], va);
            bf16x8_to_f32(vr[u][1], vb8);
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                const float pz = valid[u] ? exp2f(sc[u * GT + g] - m[g]) : 0.f;
                l[g] += pz;
#pragma unroll
                for (int i = 0; i < 8; ++i) o[g][i] = fmaf(pz, va[i], o[g][i]);
#pragma unroll
                for (int i = 0; i < 8; ++i) o[g][8 + i] = fmaf(pz, vb8[i], o[g][8 + i]);
            }
        }
    }

    // Combine the KPW lane groups (disjoint keys) of the warp.
#pragma unroll
    for (int off = C::LPK; off < 32; off <<= 1) {
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            const float mo = __shfl_xor_sync(kFull, m[g], off);
            const float lo = __shfl_xor_sync(kFull, l[g], off);
            const float M = fmaxf(m[g], mo);
            const float a = m[g] == -INFINITY ? 0.f : exp2f(m[g] - M);
            const float b = mo == -INFINITY ? 0.f : exp2f(mo - M);
            l[g] = l[g] * a + lo * b;
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const float oo = __shfl_xor_sync(kFull, o[g][i], off);
                o[g][i] = o[g][i] * a + oo * b;
            }
            m[g] = M;
        }
    }

    if (gi == 0) {
        const int slot = prefix ? split : kMaxPrefixSplits + split;
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            const size_t row = size_t(s) * P.Hq + h * P.G + rc * GT + g;
            const size_t idx = size_t(slot) * P.B * P.Hq + row;
            float4* op = reinterpret_cast<float4*>(P.ws_o + idx * D);
            op[2 * c0] = make_float4(o[g][0], o[g][1], o[g][2], o[g][3]);
            op[2 * c0 + 1] = make_float4(o[g][4], o[g][5], o[g][6], o[g][7]);
            op[2 * c1] = make_float4(o[g][8], o[g][9], o[g][10], o[g][11]);
            op[2 * c1 + 1] = make_float4(o[g][12], o[g][13], o[g][14], o[g][15]);
            if (dl == 0) P.ws_ml[idx] = make_float2(m[g], l[g]);
        }
    }
}

template <int D>
int launch_d(const AttnParams& p, bool prefix, cudaStream_t st) {
    int gt = 1;
    if (p.G % 4 == 0) gt = 4;
    else if (p.G % 2 == 0) gt = 2;
    const int nsplit = prefix ? p.nsp : p.nss;
    const long n_items = long(p.B) * p.Hkv * (p.G / gt) * nsplit;
    if (n_items == 0) return 0;
    const dim3 grid(unsigned((n_items + 3) / 4)), block(128);
    switch (gt) {
        case 4: partials_cc_kernel<D, 4><<<grid, block, 0, st>>>(p, prefix, int(n_items)); break;
        case 2: partials_cc_kernel<D, 2><<<grid, block, 0, st>>>(p, prefix, int(n_items)); break;
        default: partials_cc_kernel<D, 1><<<grid, block, 0, st>>>(p, prefix, int(n_items)); break;
    }
    return int(cudaGetLastError());
}

}  // namespace

int launch_partials_cc(const AttnParams& p, bool prefix, void* stream) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.D) {
        case 64: return launch_d<64>(p, prefix, st);
        case 128: return launch_d<128>(p, prefix, st);
        case 256: return launch_d<256>(p, prefix, st);
        default: return int(cudaErrorInvalidValue);
    }
}

}  // namespace splice
