// Generated-span pass (CUDA cores): attention of the G query rows of one
// (sequence, kv head) over that sequence's own generated-span K/V (§3: the
// decode step attends over the prompt span and the t generated entries).
//
// HBM-bound streaming kernel:
//   * persistent warps walking work items (sequence, kv head, row chunk, key
//     split) and, inside an item, blocks of 16 keys: a fixed stream per warp
//     when this pass goes first, items claimed at run time (one ahead) when
//     it runs behind the prompt-span pass, so warps that start late (on SMs
//     that pass still holds) simply take fewer; the issue cursor decodes
//     each item once and hands it to the consumer through a per-warp ring;
//   * every block's K and V rows (contiguous in the generated-span store) are
//     fetched by one bulk async copy (cp.async.bulk, mbarrier-tracked) into a
//     two-stage per-warp ring; the next block -- of this item or the next one
//     -- is in flight while the current one is computed; an item's first
//     block brings the item's query rows with it, so no item starts on a
//     load from global memory;
//   * a key row of d values is split over LPK = d / 16 lanes (16 dims each,
//     two 16-byte chunks); q . k partial sums are reduced across the LPK
//     lanes through a small shared-memory transpose (lane dl of a key group
//     ends with the full logits v = dl, dl + LPK, ..., all of query row
//     dl mod GT, read bank-conflict free), then probabilities are shared
//     back the same way; each lane sums the probabilities of its own
//     logits and the row sums are reduced once per item;
//   * packed fp32x2 FMAs (FFMA2) for both q . k and p . v;
//   * online softmax with a lazily moved reference max: the common path
//     needs no rescale and no cross-lane max; at an item's end the key
//     groups' states are combined by a reduce-scatter.
// Emits the partial state (m, l, o) of every row, like the prompt-span pass
// -- or, behind the prompt-span pass with one split of each span, merges
// the rows itself and writes the output (no merge kernel then).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"
#include "tc_ptx.cuh"

namespace splice {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr float kTau = 8.0f;
constexpr unsigned kErrWaitGs = 0x10, kErrWaitGsDrain = 0x80;

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// bf16 pair word -> (even dim, odd dim) as fp32
__device__ __forceinline__ float2 unpack2(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// Generated-span K/V is read once: the copy marks its L2 lines first to be
// evicted, so the streamed bytes do not push out the partial states the
// merge reads right after.
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ unsigned ld_relaxed_gpu(const unsigned* p) {
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p));
    return v;
}

// The merge of a row's two partial states -- the prompt-span pass's (when
// has_span) and this pass's -- with a ZERO span's closed form, in exactly
// the operations and order of the merge kernel for a row of at most two
// states (merge_row.cuh): the same bits.  Returns the factor of the
// weighted sum (0 for a row with nothing live) and the two weights.
__device__ __forceinline__ float merge_two_weights(bool has_span, float2 ml_span, float m_gen, float l_gen,
                                                   bool zero_span, int n_zero, float* w_span, float* w_gen) {
    const bool live_s = has_span && ml_span.y > 0.f, live_g = l_gen > 0.f;
    float M = fmaxf(live_s ? ml_span.x : -INFINITY, live_g ? m_gen : -INFINITY);
    if (zero_span) M = fmaxf(M, 0.f);
    *w_span = live_s ? exp2f(ml_span.x - M) : 0.f;
    *w_gen = live_g ? exp2f(m_gen - M) : 0.f;
    float den = __fadd_rn(has_span ? __fmul_rn(*w_span, ml_span.y) : 0.f, __fmul_rn(*w_gen, l_gen));
    if (zero_span) den = fmaf(float(n_zero), exp2f(0.f - M), den);
    return den > 0.f ? 1.f / den : 0.f;
}

__device__ __forceinline__ float merge_two(bool has_span, float w_span, float o_span, float w_gen, float o_gen,
                                           float inv) {
    float acc = 0.f;
    if (has_span && w_span != 0.f) acc = fmaf(w_span, o_span, acc);
    if (w_gen != 0.f) acc = fmaf(w_gen, o_gen, acc);
    return __fmul_rn(acc, inv);
}

// The same without a cache hint: the query rows are read again by the
// prompt-span pass of the call.
__device__ __forceinline__ void bulk_copy_plain(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

// Items a warp may leave unmerged until its end (with P.gs_merge): those
// that end before the prompt-span pass has completed.
constexpr int kPend = 8;

template <int D, int GT>
struct GS {
    static constexpr int LPK = D / 16;              // lanes per key
    static constexpr int KPW = 32 / LPK;            // key groups per warp
    static constexpr int BK = 16;                   // keys per block
    static constexpr int U = BK / KPW;              // keys per group per block
    static constexpr int NV = U * GT;               // logits per group per block
    static constexpr int VPL = NV >= LPK ? NV / LPK : 1;   // logits reduced by each lane
    static constexpr int WARPS = D == 256 ? 2 : 4;
    static constexpr int RED = NV + 4;              // padded floats per lane in the reduce buffer
    // floats per key group in the reduce buffer: a multiple of 32 plus LPK,
    // so the LPK partials of logit v of the KPW groups land in 32 distinct banks
    static constexpr int GSTRIDE = (LPK * RED + 31) / 32 * 32 + LPK;
    static constexpr int VPL_LIVE = NV >= LPK ? LPK : NV;   // lanes of a group holding distinct logits
    static constexpr uint32_t ROW = D * 2;          // bytes of one key row
    static constexpr uint32_t STAGE = BK * ROW * 2; // K + V block
    // per-warp shared memory: 2 stages, reduce buffer, probability pairs, 2 barriers
    static constexpr uint32_t OFF_RED = 2 * STAGE;
    static constexpr uint32_t OFF_PP = OFF_RED + KPW * GSTRIDE * 4;
    static constexpr uint32_t OFF_BAR = OFF_PP + KPW * NV * 8;
    static constexpr uint32_t OFF_TAKEN = OFF_BAR + 16;       // [4] items (decoded) in the order the issue cursor took them
    static constexpr uint32_t QROWS = GT * D * 2;             // the GT query rows of one item
    static constexpr uint32_t OFF_Q = OFF_TAKEN + 4 * 32;     // [2] query rows, brought with each item's first block
    static constexpr uint32_t OFF_PEND = OFF_Q + 2 * QROWS;   // [kPend] items whose merge waits for the warp's end
    static constexpr uint32_t PER_WARP = (OFF_PEND + kPend * 4 + 127) / 128 * 128;
    static constexpr uint32_t SMEM = WARPS * PER_WARP;
    static_assert(NV % 4 == 0 || NV < 4, "reduce layout");
    static_assert(NV < LPK || NV == VPL * LPK, "every logit of a group owned by one lane");
    static_assert(LPK % GT == 0, "the logits of a lane belong to one query row");
};

// n / d for 0 <= n < 2^31 by a multiply and a shift, for a divisor fixed
// per launch (Granlund and Montgomery, "Division by invariant integers using
// multiplication", 1994, the round-up method): with s = ceil(log2 d) and
// m = floor(2^32 (2^s - d) / d) + 1, n / d = (umulhi(n, m) + n) >> s; the
// sum stays below 2^32 because umulhi(n, m) < n < 2^31.
struct FastDiv {
    uint32_t d, m, s;
    __device__ explicit FastDiv(int divisor) : d(uint32_t(divisor)), m(1), s(0) {
        while ((1u << s) < d) ++s;
        m = uint32_t((((uint64_t(1) << s) - d) << 32) / d + 1);
    }
    __device__ __forceinline__ int div(int n) const { return int((__umulhi(uint32_t(n), m) + uint32_t(n)) >> s); }
};

struct ItemDivs {
    FastDiv nss, n_rc, hkv;
};

// One work item: where its rows and keys are.  The issue cursor decodes
// each item once and hands it to the consumer through the warp's ring
// (eight ints, idx -1 for the end of the walk).
struct Item {
    int idx, s, h, rc, split, k0, k1, nblk;
};

// Work item idx = ((sequence * Hkv + kv head) * row chunks + row chunk) *
// splits + key split.
__device__ __forceinline__ void item_of(const AttnParams& P, const ItemDivs& dv, int idx, Item& it) {
    it.idx = idx;
    int rem = dv.nss.div(idx);
    it.split = idx - rem * P.nss;
    const int sh = dv.n_rc.div(rem);
    it.rc = rem - sh * int(dv.n_rc.d);
    it.s = dv.hkv.div(sh);
    it.h = sh - it.s * P.Hkv;
    it.k0 = P.s_lo + it.split * P.s_chunk;
    it.k1 = min(P.s_hi, it.k0 + P.s_chunk);
    it.nblk = it.k1 > it.k0 ? (it.k1 - it.k0 + 15) / 16 : 0;
}

// Offset (in elements) of the generated-span K/V rows of (sequence, kv head)
// at this layer.
template <int D>
__device__ __forceinline__ size_t span_base(const AttnParams& P, int s, int h) {
    return ((size_t(s) * P.N + P.layer) * P.Hkv + h) * size_t(P.T) * D;
}

template <int D, int GT>
__global__ void __launch_bounds__(GS<D, GT>::WARPS * 32)
    gs_kernel(const AttnParams P, int n_items, int sm_count) {
    using C = GS<D, GT>;
    extern __shared__ __align__(128) uint8_t smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // The call's first pass: launched as a programmatic dependent of
    // whatever precedes it on the stream, this grid may start before that
    // work has finished, so it waits for it (its writes visible) before
    // reading or writing anything.  Only then may the pass queued behind it
    // launch: the prompt-span pass reads the queries and the prompt stores
    // without a wait of its own, and it reads nothing this grid writes, so it
    // may take the SMs this grid's last CTAs leave.  (Behind the prompt-span
    // pass instead, that pass has waited before it let this grid launch, and
    // this grid reads what it writes only after that pass's completion flag,
    // with P.gs_merge; see the end of the kernel.)  No-ops for a plain
    // launch.
    if (!P.gs_after_prefix) {
        asm volatile("griddepcontrol.wait;" ::: "memory");
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    }
    uint8_t* ws = smem + warp * C::PER_WARP;
    const uint32_t wbase = tc::smem_u32(ws);
    const uint32_t bar0 = wbase + C::OFF_BAR;
    float* red = reinterpret_cast<float*>(ws + C::OFF_RED);
    float2* pp = reinterpret_cast<float2*>(ws + C::OFF_PP);
    int4* ring = reinterpret_cast<int4*>(ws + C::OFF_TAKEN);
    int* pend = reinterpret_cast<int*>(ws + C::OFF_PEND);
    int npend = 0;

    const int gi = lane / C::LPK, dl = lane % C::LPK;
    const int g_mine = dl % GT;
    const int c0 = dl, c1 = dl + C::LPK;
    volatile int abort_flag = 0;

    if (lane == 0) {
        tc::mbar_init(bar0, 1);
        tc::mbar_init(bar0 + 8, 1);
        tc::fence_mbar_init();
    }
    __syncwarp();

    // ---- work items: the warp of rank r starts on item r.  As the call's
    // first pass (all warps start together) it then walks items r + k *
    // (warps of the grid): the extra items of an uneven share land on the
    // lowest ranks, so the other SMs come free whole and early for the
    // prompt-span pass queued behind.  Behind the prompt-span pass (CTAs
    // start as that pass's CTAs leave) every later item is claimed from the
    // launch-wide counter (numbered from the grid's warp count on), one
    // ahead: lane 0 holds the claim in flight, whose value is needed only
    // when the next item starts (the prompt-span pass clears the counter
    // before this grid can launch) ----
    const unsigned nwarps = gridDim.x * C::WARPS;
    // The warps' ranks.  With the prompt-span pass queued behind, SM-major
    // when the grid is whole waves of sm_count CTAs: the first wave's CTAs
    // land on distinct SMs and each later wave stacks one more CTA on each
    // in the same order, so CTAs b, b + sm_count, ... share an SM and get
    // consecutive ranks -- the extra items of an uneven share then fill
    // whole SMs, and the others come free together for that pass.  With
    // nothing queued behind, CTA-major, which spreads the extra items over
    // the SMs.
    int rank = int(blockIdx.x) * C::WARPS + warp;
    if (P.prefix_after_gs && sm_count > 0 && gridDim.x % unsigned(sm_count) == 0) {
        const int cps = int(gridDim.x) / sm_count;
        rank = ((int(blockIdx.x) % sm_count) * cps + int(blockIdx.x) / sm_count) * C::WARPS + warp;
    }
    const int first_item = rank;
    const bool claims = P.gs_after_prefix != 0;
    unsigned claim = unsigned(first_item) + nwarps;
    // d = 256 (fewer, longer items per warp): the claim goes out two blocks
    // before the item's end instead, so no warp holds an item it will not
    // start soon (about +1% on a Gemma-3-4B-shaped sweep; for d <= 128 the
    // same code measured slower).
    constexpr bool kLateClaim = D == 256;
    bool have_claim = !claims || !kLateClaim;
    if (!kLateClaim && claims && lane == 0) claim = nwarps + atomicAdd(P.sched + 2, 1u);
    auto request = [&]() {
        if (!have_claim) {
            if (lane == 0) claim = nwarps + atomicAdd(P.sched + 2, 1u);
            have_claim = true;
        }
    };
    auto next_item = [&]() -> int {
        if constexpr (kLateClaim) {
            request();   // an item too short for the early request
            const int i = int(__shfl_sync(kFull, claim, 0));
            if (claims) {
                have_claim = false;
            } else {
                claim += nwarps;
            }
            return i < n_items ? i : -1;
        } else {
            const int i = int(__shfl_sync(kFull, claim, 0));
            if (i >= n_items) return -1;
            if (claims) {
                if (lane == 0) claim = nwarps + atomicAdd(P.sched + 2, 1u);
            } else {
                claim += nwarps;
            }
            return i;
        }
    };

    // ---- issue cursor: walks (item, block) in claim order and records every
    // item it takes, decoded (then the end, idx -1), for the consumer.  It
    // runs two blocks ahead and every item has a block (the host keeps at
    // least 64 keys per split), so it is at most two items ahead ----
    const ItemDivs dv{FastDiv(P.nss), FastDiv(P.G / GT), FastDiv(P.Hkv)};
    Item iss;
    int iss_idx = first_item < n_items ? first_item : -1, iss_b = 0, recorded = 0;
    bool iss_ok = false;
    auto record = [&](const Item& e) {
        if (lane == 0) {
            ring[2 * (recorded & 3)] = make_int4(e.idx, e.s, e.h, e.rc);
            ring[2 * (recorded & 3) + 1] = make_int4(e.split, e.k0, e.k1, e.nblk);
        }
        ++recorded;
    };
    auto seek = [&]() {   // the first block at or after item iss_idx
        iss_ok = false;
        while (iss_idx >= 0) {
            item_of(P, dv, iss_idx, iss);
            record(iss);
            if (iss.nblk > 0) {
                iss_ok = true;
                return;
            }
            iss_idx = next_item();
        }
        iss.idx = -1;
        record(iss);
    };
    seek();
    int issued = 0, iss_items = 0;
    const uint64_t pol = l2_evict_first_policy();
    size_t iss_base = iss_ok ? span_base<D>(P, iss.s, iss.h) : 0;
    auto issue_next = [&]() {
        if (!iss_ok) return;
        const int stg = issued & 1;
        // an item's first block also brings the item's GT query rows
        // (contiguous in q) into the item's query buffer
        const bool first = iss_b == 0;
        const int j = iss.k0 + iss_b * 16;
        int nk = min(16, iss.k1 - j);
        // fused append: entry step - 1 (the block's last row) is not in the
        // store yet; the consumer writes that row of the stage from registers
        if (P.fuse_append && j + nk == P.s_hi) --nk;
        const uint32_t bytes = uint32_t(nk) * C::ROW;
        if (lane == 0) {
            const uint32_t dst = wbase + stg * C::STAGE;
            tc::mbar_arrive_expect_tx(bar0 + 8 * stg, 2 * bytes + (first ? C::QROWS : 0u));
            if (first)
                bulk_copy_plain(wbase + C::OFF_Q + (iss_items & 1) * C::QROWS,
                                P.q + (size_t(iss.s) * P.Hq + iss.h * P.G + iss.rc * GT) * D, C::QROWS, bar0 + 8 * stg);
            if (bytes) {
                bulk_copy(dst, P.ks + iss_base + size_t(j) * D, bytes, bar0 + 8 * stg, pol);
                bulk_copy(dst + C::BK * C::ROW, P.vs + iss_base + size_t(j) * D, bytes, bar0 + 8 * stg, pol);
            }
        }
        ++issued;
        if (first) ++iss_items;
        if constexpr (kLateClaim) {
            if (claims && iss_b + 2 >= iss.nblk) request();
        }
        if (++iss_b >= iss.nblk) {
            iss_b = 0;
            iss_idx = next_item();
            seek();
            if (iss_ok) iss_base = span_base<D>(P, iss.s, iss.h);
        }
    };
    issue_next();
    issue_next();

    int consumed = 0, cons_items = 0;
    bool ok = true;
    bool ps_ready = false;   // the prompt-span pass's states are complete and visible
    // This lane's dims after the key groups' reduce-scatter (below): F of
    // the 16 it holds, from index `kept` on (round r keeps the upper half
    // when bit r of gi is set); dims 8 c0 .. 8 c0 + 7 are the first 8 of
    // the 16, 8 c1 .. 8 c1 + 7 the last 8.
    constexpr int F = 16 / C::KPW;
    // the merge path is built where its prompt-span states fit in registers
    constexpr bool kCanMerge = GT * F <= 16;
    int kept = 0;
#pragma unroll
    for (int r = 0; (C::LPK << r) < 32; ++r)
        if ((gi >> r) & 1) kept += 8 >> r;
    const int dim0 = kept < 8 ? 8 * c0 + kept : 8 * c1 + (kept - 8);
    for (int taken = 0; ok; ++taken) {
        __syncwarp();
        const int4 e0 = ring[2 * (taken & 3)];
        if (e0.x < 0) break;
        const int4 e1 = ring[2 * (taken & 3) + 1];
        const Item it{e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
        // merges in this pass: the rows' source (a ZERO row needs no
        // prompt-span state) and, until it has been seen set, the prompt-span
        // pass's completion flag, read now and used at the item's end
        unsigned code = 0, poll = 0;
        if (kCanMerge && P.gs_merge) {
            code = P.src[it.s];
            if (!ps_ready) poll = ld_relaxed_gpu(P.sched + 4);
        }
        // q rows of this item, pre-scaled into log2 units, as dim pairs: in
        // the item's query buffer once its first block has landed
        float2 q2[GT][8];
        if (it.nblk > 0) {
            const bool got = tc::mbar_wait(bar0 + 8 * (consumed & 1), uint32_t(consumed >> 1) & 1u, &abort_flag,
                                           P.err, kErrWaitGs);
            if (!__all_sync(kFull, got)) {
                ok = false;
                break;
            }
        }
        const uint8_t* qsm = ws + C::OFF_Q + (cons_items & 1) * C::QROWS;
        if (it.nblk > 0) ++cons_items;
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            const uint4* qr = reinterpret_cast<const uint4*>(qsm + g * D * 2);
            const uint4 a = qr[c0], b = qr[c1];
            const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const float2 f = unpack2(w[i]);
                q2[g][i] = make_float2(f.x * P.scale_log2, f.y * P.scale_log2);
            }
        }
        // m: every row's reference max (the same in every lane of a key
        // group); m_mine: that of row g_mine, the row of this lane's logits;
        // l_mine: this lane's share of row g_mine's sum
        float m[GT];
        float2 o2[GT][8];
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            m[g] = -INFINITY;
#pragma unroll
            for (int i = 0; i < 8; ++i) o2[g][i] = make_float2(0.f, 0.f);
        }
        float m_mine = -INFINITY, l_mine = 0.f;
        // fused append: this item's split ends at the step's own entry (step
        // - 1), which comes from the new K/V rows, loaded now (lanes take
        // 16-byte chunks: the K row's D / 8, then the V row's)
        constexpr int NCH = D / 4;                       // 16-byte chunks of the K and V rows
        constexpr int CPL = NCH >= 32 ? NCH / 32 : 1;    // chunks per lane
        const bool tail = P.fuse_append && it.k1 == P.s_hi && it.nblk > 0;
        uint4 nkv[CPL];
        if (tail) {
            const size_t rowc = (size_t(it.s) * P.Hkv + it.h) * (D / 8);
#pragma unroll
            for (int i = 0; i < CPL; ++i) {
                const int c = lane + 32 * i;
                if (c < NCH)
                    nkv[i] = c < D / 8 ? reinterpret_cast<const uint4*>(P.kn)[rowc + c]
                                       : reinterpret_cast<const uint4*>(P.vn)[rowc + c - D / 8];
            }
        }

        for (int b = 0; b < it.nblk; ++b) {
            const int stg = consumed & 1;
            const bool got = tc::mbar_wait(bar0 + 8 * stg, uint32_t(consumed >> 1) & 1u, &abort_flag, P.err, kErrWaitGs);
            if (!__all_sync(kFull, got)) {
                ok = false;
                break;
            }
            uint8_t* kst = ws + stg * C::STAGE;
            uint8_t* vst = kst + C::BK * C::ROW;
            const int jb = it.k0 + b * 16;
            if (tail && b == it.nblk - 1) {
                // the step's own entry: its row of the stage from registers,
                // and (once per (sequence, kv head)) into the store
                const int rj = P.s_hi - 1 - jb;
                const size_t ent = ((size_t(it.s) * P.N + P.layer) * P.Hkv + it.h) * size_t(P.T) + (P.s_hi - 1);
#pragma unroll
                for (int i = 0; i < CPL; ++i) {
                    const int c = lane + 32 * i;
                    if (c < NCH) {
                        const bool isk = c < D / 8;
                        const int cc = isk ? c : c - D / 8;
                        *reinterpret_cast<uint4*>((isk ? kst : vst) + rj * C::ROW + cc * 16) = nkv[i];
                        if (it.rc == 0)
                            reinterpret_cast<uint4*>(isk ? P.ks_w : P.vs_w)[ent * (D / 8) + cc] = nkv[i];
                    }
                }
                __syncwarp();
            }

            // ---- partial q . k over this lane's 16 dims ----
            float dot[C::NV];
#pragma unroll
            for (int u = 0; u < C::U; ++u) {
                const int kb = u * C::KPW + gi;
                const uint4 ka = *reinterpret_cast<const uint4*>(kst + kb * C::ROW + c0 * 16);
                const uint4 kc = *reinterpret_cast<const uint4*>(kst + kb * C::ROW + c1 * 16);
                const uint32_t w[8] = {ka.x, ka.y, ka.z, ka.w, kc.x, kc.y, kc.z, kc.w};
                float2 k2[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) k2[i] = unpack2(w[i]);
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    float2 acc = __fmul2_rn(q2[g][0], k2[0]);
#pragma unroll
                    for (int i = 1; i < 8; ++i) acc = __ffma2_rn(q2[g][i], k2[i], acc);
                    dot[u * GT + g] = acc.x + acc.y;
                }
            }
            // ---- transpose-reduce across the LPK lanes of the group ----
            float* gred = red + gi * C::GSTRIDE;
            float* myred = gred + dl * C::RED;
            if constexpr (C::NV % 4 == 0) {
#pragma unroll
                for (int v = 0; v < C::NV; v += 4)
                    *reinterpret_cast<float4*>(myred + v) = make_float4(dot[v], dot[v + 1], dot[v + 2], dot[v + 3]);
            } else {
#pragma unroll
                for (int v = 0; v < C::NV; ++v) myred[v] = dot[v];
            }
            __syncwarp();
            float sv[C::VPL];
            bool need = false;
#pragma unroll
            for (int i = 0; i < C::VPL; ++i) {
                const int v = (dl + C::LPK * i) % C::NV;
                float part[C::LPK];
#pragma unroll
                for (int q = 0; q < C::LPK; ++q) part[q] = gred[q * C::RED + v];
#pragma unroll
                for (int w = C::LPK / 2; w > 0; w >>= 1) {
#pragma unroll
                    for (int q = 0; q < w; ++q) part[q] += part[q + w];
                }
                const int u = v / GT;
                const bool valid = jb + u * C::KPW + gi < it.k1;
                sv[i] = valid ? part[0] : -INFINITY;
                need |= sv[i] > m_mine + kTau;
            }
            if (__any_sync(kFull, need)) {
                // rare: some row's reference max moves; share every logit of
                // the group and recompute the per-row block maxima
                __syncwarp();
#pragma unroll
                for (int i = 0; i < C::VPL; ++i) gred[(dl + C::LPK * i) % C::NV] = sv[i];
                __syncwarp();
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    float mb = -INFINITY;
#pragma unroll
                    for (int u = 0; u < C::U; ++u) mb = fmaxf(mb, gred[u * GT + g]);
                    if (mb > m[g] + kTau) {
                        const float alpha = ex2(m[g] - mb);
                        if (g == g_mine) l_mine *= alpha;
                        const float2 a2 = make_float2(alpha, alpha);
#pragma unroll
                        for (int i = 0; i < 8; ++i) o2[g][i] = __fmul2_rn(o2[g][i], a2);
                        m[g] = mb;
                    }
                }
#pragma unroll
                for (int g = 0; g < GT; ++g)
                    if (g == g_mine) m_mine = m[g];
            }
            // ---- probabilities, shared back as (p, p) pairs ----
            __syncwarp();
            float2* mypp = pp + gi * C::NV;
            const float mg = m_mine == -INFINITY ? 0.f : m_mine;
#pragma unroll
            for (int i = 0; i < C::VPL; ++i) {
                const float p = ex2(sv[i] - mg);
                l_mine += p;
                if (C::NV >= C::LPK || dl < C::NV) mypp[(dl + C::LPK * i) % C::NV] = make_float2(p, p);
            }
            __syncwarp();
            float2 p2[C::NV];
#pragma unroll
            for (int v = 0; v < C::NV; v += 2) {
                const float4 t = *reinterpret_cast<const float4*>(mypp + v);
                p2[v] = make_float2(t.x, t.y);
                if (v + 1 < C::NV) p2[v + 1] = make_float2(t.z, t.w);
            }
            // ---- o += p . v over this lane's 16 dims ----
#pragma unroll
            for (int u = 0; u < C::U; ++u) {
                const int kb = u * C::KPW + gi;
                if (jb + kb < it.k1) {
                    const uint4 va = *reinterpret_cast<const uint4*>(vst + kb * C::ROW + c0 * 16);
                    const uint4 vc = *reinterpret_cast<const uint4*>(vst + kb * C::ROW + c1 * 16);
                    const uint32_t w[8] = {va.x, va.y, va.z, va.w, vc.x, vc.y, vc.z, vc.w};
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const float2 v2 = unpack2(w[i]);
#pragma unroll
                        for (int g = 0; g < GT; ++g) o2[g][i] = __ffma2_rn(p2[u * GT + g], v2, o2[g][i]);
                    }
                }
            }
            // stage free: every lane is done reading it
            __syncwarp();
            tc::fence_proxy_async_smem();
            ++consumed;
            issue_next();
        }
        if (!ok) break;

        // ---- merge here?  Always for a ZERO row; for the others once the
        // prompt-span pass has completed, whose states are fetched now (this
        // lane's dims of every row), under the reduction below.  An item
        // that ends before then writes its partial state and is merged at
        // the warp's end (up to kPend of them; past that the warp waits
        // for the prompt-span grid here) ----
        bool merge_here = false;
        const bool has_span = code != SPLICE_SRC_ZERO;
        float2 ml_span[GT];
        float o_span[GT][F];
        if (kCanMerge && P.gs_merge) {
            if (!ps_ready && __all_sync(kFull, poll != 0u)) {
                asm volatile("fence.acq_rel.gpu;" ::: "memory");
                ps_ready = true;
            }
            merge_here = !has_span || ps_ready;
            if (!merge_here) {
                if (npend < kPend) {
                    if (lane == 0) pend[npend] = it.idx;
                    ++npend;
                } else {
                    asm volatile("griddepcontrol.wait;" ::: "memory");
                    ps_ready = true;
                    merge_here = true;
                }
            }
            if (merge_here && has_span) {
#pragma unroll
                for (int g = 0; g < GT; ++g) {
                    const size_t row = size_t(it.s) * P.Hq + it.h * P.G + it.rc * GT + g;   // split 0's slot
                    ml_span[g] = __ldcg(P.ws_ml + row);
                    const float* sp = P.ws_o + row * D + dim0;
                    if constexpr (F == 2) {
                        const float2 t = __ldcg(reinterpret_cast<const float2*>(sp));
                        o_span[g][0] = t.x;
                        o_span[g][1] = t.y;
                    } else {
#pragma unroll
                        for (int k = 0; k < F; k += 4) {
                            const float4 t = __ldcg(reinterpret_cast<const float4*>(sp + k));
                            o_span[g][k] = t.x;
                            o_span[g][k + 1] = t.y;
                            o_span[g][k + 2] = t.z;
                            o_span[g][k + 3] = t.w;
                        }
                    }
                }
            }
        }

        // ---- row sums of the group: the lanes holding distinct logits ----
        float l[GT];
#pragma unroll
        for (int g = 0; g < GT; ++g) {
            float x = (g == g_mine && dl < C::VPL_LIVE) ? l_mine : 0.f;
#pragma unroll
            for (int off = 1; off < C::LPK; off <<= 1) x += __shfl_xor_sync(kFull, x, off);
            l[g] = x;
        }

        // ---- combine the KPW key groups of the warp, a reduce-scatter: round
        // r pairs group gi with group gi ^ 2^r, both rescale to the pair's
        // max, and each keeps the half of its dims that its partner sends
        // it; after log2(KPW) rounds every lane holds F = 16 / KPW dims of
        // every row, summed over the groups, and m, l of every row ----
        float v[GT][16];
#pragma unroll
        for (int g = 0; g < GT; ++g) {
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                v[g][2 * i] = o2[g][i].x;
                v[g][2 * i + 1] = o2[g][i].y;
            }
        }
#pragma unroll
        for (int r = 0; (C::LPK << r) < 32; ++r) {
            const int off = C::LPK << r, W = 16 >> r;
            const bool hi = (gi >> r) & 1;
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                const float mo = __shfl_xor_sync(kFull, m[g], off);
                const float lo = __shfl_xor_sync(kFull, l[g], off);
                const float M = fmaxf(m[g], mo);
                const float a = m[g] == -INFINITY ? 0.f : ex2(m[g] - M);
                const float bb = mo == -INFINITY ? 0.f : ex2(mo - M);
                l[g] = l[g] * a + lo * bb;
#pragma unroll
                for (int k = 0; k < W / 2; ++k) {
                    const float send = hi ? v[g][k] : v[g][W / 2 + k];
                    const float keep = hi ? v[g][W / 2 + k] : v[g][k];
                    const float recv = __shfl_xor_sync(kFull, send, off);
                    v[g][k] = keep * a + recv * bb;
                }
                m[g] = M;
            }
        }
        if (kCanMerge && merge_here) {
            // the output
            const bool zero_span = !has_span && P.p_hi > P.p_lo;
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                const size_t row = size_t(it.s) * P.Hq + it.h * P.G + it.rc * GT + g;
                // the row's (m, l) as lane 0 would store it: the lanes' row
                // sums can differ in the last bit (each lane adds its pair's
                // two terms in its own order)
                const float mg = __shfl_sync(kFull, m[g], 0), lg = __shfl_sync(kFull, l[g], 0);
                float w_span, w_gen;
                const float inv = merge_two_weights(has_span, has_span ? ml_span[g] : make_float2(-INFINITY, 0.f),
                                                    mg, lg, zero_span, P.p_hi - P.p_lo, &w_span, &w_gen);
                float r[F];
#pragma unroll
                for (int k = 0; k < F; ++k)
                    r[k] = merge_two(has_span, w_span, has_span ? o_span[g][k] : 0.f, w_gen, v[g][k], inv);
                float* op = P.out + row * D + dim0;
                if constexpr (F == 2) {
                    *reinterpret_cast<float2*>(op) = make_float2(r[0], r[1]);
                } else {
#pragma unroll
                    for (int k = 0; k < F; k += 4)
                        *reinterpret_cast<float4*>(op + k) = make_float4(r[k], r[k + 1], r[k + 2], r[k + 3]);
                }
            }
        } else {
            const int slot = kMaxPrefixSplits + it.split;
#pragma unroll
            for (int g = 0; g < GT; ++g) {
                const size_t row = size_t(it.s) * P.Hq + it.h * P.G + it.rc * GT + g;
                const size_t idx2 = size_t(slot) * P.B * P.Hq + row;
                float* op = P.ws_o + idx2 * D + dim0;
                if constexpr (F == 2) {
                    *reinterpret_cast<float2*>(op) = make_float2(v[g][0], v[g][1]);
                } else {
#pragma unroll
                    for (int k = 0; k < F; k += 4)
                        *reinterpret_cast<float4*>(op + k) = make_float4(v[g][k], v[g][k + 1], v[g][k + 2], v[g][k + 3]);
                }
                if (lane == 0) P.ws_ml[idx2] = make_float2(m[g], l[g]);
            }
        }
    }
    // Copies still in flight (only after an abort: at most the two of the
    // ring) must land before the warp's shared memory is given up.  A bulk
    // copy from global memory waits on nothing else on the GPU, so it lands;
    // the long bound only keeps a broken memory system from holding the CTA
    // forever, and a drain that runs out records its own error bit.
    for (; consumed < issued; ++consumed) {
        volatile int no_abort = 0;
        tc::mbar_wait(bar0 + 8 * (consumed & 1), uint32_t(consumed >> 1) & 1u, &no_abort, P.err, kErrWaitGsDrain,
                      10000000000ull);
    }
    if (P.gs_after_prefix) {
        // Behind the prompt-span pass: this grid's completion must imply that
        // pass's, so the merge queued behind this grid sees both (with
        // P.gs_merge no merge is queued: this grid writes every output).
        // Then the work behind may launch (the merge waits for this whole
        // grid before it reads anything); every CTA of this grid is running
        // by the time all of them have signalled, so those CTAs never hold
        // an SM it still needs.
        asm volatile("griddepcontrol.wait;" ::: "memory");
        // The items left unmerged: the prompt-span states are complete and
        // visible now; this warp's own partial states are re-read (the same
        // bits it stored) and merged as at an item's end.
        if constexpr (kCanMerge) {
            if (P.gs_merge && npend > 0) {
                __syncwarp();
                for (int k = 0; k < npend; ++k) {
                    Item it;
                    item_of(P, dv, pend[k], it);
#pragma unroll
                    for (int g = 0; g < GT; ++g) {
                        const size_t row = size_t(it.s) * P.Hq + it.h * P.G + it.rc * GT + g;
                        const size_t gen = size_t(kMaxPrefixSplits) * P.B * P.Hq + row;
                        const float2 ml_gen = __ldcg(P.ws_ml + gen), ml_span = __ldcg(P.ws_ml + row);
                        float og[F], os[F];
#pragma unroll
                        for (int j = 0; j < F; j += 2) {
                            const float2 a = __ldcg(reinterpret_cast<const float2*>(P.ws_o + gen * D + dim0 + j));
                            const float2 b = __ldcg(reinterpret_cast<const float2*>(P.ws_o + row * D + dim0 + j));
                            og[j] = a.x;
                            og[j + 1] = a.y;
                            os[j] = b.x;
                            os[j + 1] = b.y;
                        }
                        float w_span, w_gen;
                        const float inv = merge_two_weights(true, ml_span, ml_gen.x, ml_gen.y, false, 0, &w_span, &w_gen);
                        float* op = P.out + row * D + dim0;
#pragma unroll
                        for (int j = 0; j < F; j += 2)
                            *reinterpret_cast<float2*>(op + j) = make_float2(merge_two(true, w_span, os[j], w_gen, og[j], inv),
                                                                             merge_two(true, w_span, os[j + 1], w_gen,
                                                                                       og[j + 1], inv));
                    }
                }
            }
        }
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    }
    // (Run-time claims: the prompt-span pass ahead of this grid cleared the
    // item counter before this grid could launch.)
}

template <int D, int GT>
int launch_gs_t(const AttnParams& p, int n_items, cudaStream_t st, bool overlap_previous) {
    using C = GS<D, GT>;
    static int blocks_per_sm = 0, sms = 0;
    if (!blocks_per_sm) {
        cudaFuncSetAttribute(gs_kernel<D, GT>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks_per_sm, gs_kernel<D, GT>, C::WARPS * 32, C::SMEM);
        if (blocks_per_sm < 1) blocks_per_sm = 1;
    }
    const long want = (long(n_items) + C::WARPS - 1) / C::WARPS;
    const long cap = long(blocks_per_sm) * sms;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(want < cap ? want : cap));
    cfg.blockDim = dim3(C::WARPS * 32);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = overlap_previous ? 1 : 0;
    return int(cudaLaunchKernelEx(&cfg, gs_kernel<D, GT>, p, n_items, sms));
}

}  // namespace

int generated_span_resident_warps(int d) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // two 4-warp CTAs per SM (d <= 128), three 2-warp CTAs per SM (d = 256)
    return sms * (d == 256 ? 6 : 8);
}

bool generated_span_can_merge(int d, int G) {
    const int gt = G % 4 == 0 ? 4 : (G % 2 == 0 ? 2 : 1);
    return gt * d <= 512;   // GT * F <= 16 in gs_kernel, F = d / 32
}

int launch_generated_span(const AttnParams& p, void* stream, bool overlap_previous) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int gt = p.G % 4 == 0 ? 4 : (p.G % 2 == 0 ? 2 : 1);
    const long n_items = long(p.B) * p.Hkv * (p.G / gt) * p.nss;
    if (n_items == 0) return 0;
    switch (p.D * 8 + gt) {
        case 64 * 8 + 1: return launch_gs_t<64, 1>(p, int(n_items), st, overlap_previous);
        case 64 * 8 + 2: return launch_gs_t<64, 2>(p, int(n_items), st, overlap_previous);
        case 64 * 8 + 4: return launch_gs_t<64, 4>(p, int(n_items), st, overlap_previous);
        case 128 * 8 + 1: return launch_gs_t<128, 1>(p, int(n_items), st, overlap_previous);
        case 128 * 8 + 2: return launch_gs_t<128, 2>(p, int(n_items), st, overlap_previous);
        case 128 * 8 + 4: return launch_gs_t<128, 4>(p, int(n_items), st, overlap_previous);
        case 256 * 8 + 1: return launch_gs_t<256, 1>(p, int(n_items), st, overlap_previous);
        case 256 * 8 + 2: return launch_gs_t<256, 2>(p, int(n_items), st, overlap_previous);
        case 256 * 8 + 4: return launch_gs_t<256, 4>(p, int(n_items), st, overlap_previous);
        default: return int(cudaErrorInvalidValue);
    }
}

}  // namespace splice
