// Tensor-core prompt-span pass (tcgen05 + TMEM, TMA-fed), persistent.
//
// Every sequence that reads the same (prompt, source) span at a (layer,
// step) -- a group of the descriptor's table -- shares that span's K/V.  For
// one kv head h, the G query rows of every sequence of the group are stacked
// into 128-row tiles, so Q K^T and P V over the span are dense contractions
// (M = 128 stacked rows).  A work item is one (row tile, kv head, key split);
// each CTA walks a fixed stream of items:
//
//   warp 0        TMA producer: K and V blocks of the item's span -> a
//                 two-stage smem ring, running ahead across item boundaries
//   warp 1        MMA issuer (one lane): S = Q K^T into TMEM (two buffers);
//                 O += P V with P read from TMEM; O double-buffered in TMEM
//                 when it fits; owns the TMEM allocation
//   warp 2        Q gather: the tile's query rows -> smem (double-buffered),
//                 one item ahead
//   warps 3..10   softmax, two warpgroups: each thread owns one row and one
//                 half of every key block; the halves trade block maxima
//                 through smem, share one lazily moved reference max, write
//                 P (bf16) over their own half of S in TMEM, rescale their
//                 half of O when the reference moves, and at the item's end
//                 write the row's partial state (m, l, o) to the workspace.
//
// The merge kernel combines these partials with those of the generated span
// (and the ZERO closed form).  Every wait is bounded: a wait that runs out
// sets a CTA abort flag and an error bit in the descriptor's error word; all
// roles then leave their loops, outstanding copies and MMAs are waited for
// (bounded), TMEM is freed and the CTA exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"
#include "tc_ptx.cuh"

namespace splice {
namespace {

constexpr int kRows = 128;          // MMA M
constexpr int kWarps = 11;
constexpr int kThreads = kWarps * 32;
constexpr int kSoftmaxThreads = 256;
constexpr uint32_t kTmemCols = 512;
constexpr float kTau = 8.0f;        // lazy rescale threshold, log2 units

constexpr unsigned kErrWaitProducer = 0x1, kErrWaitMma = 0x2, kErrWaitSoftmax = 0x4, kErrWaitDrain = 0x8,
                   kErrWaitQ = 0x20;

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// A = P (bf16, in TMEM), B = V (smem descriptor): D[tmem] (+)= A * B.
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]),
        "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}

template <int D>
struct Cfg {
    static constexpr int BN = D == 256 ? 64 : 128;          // keys per block
    static constexpr int HALF = BN / 2;                     // keys per softmax thread per block
    static constexpr int STAGES = 2;
    static constexpr int KB = D / 64;                         // 64-wide K blocks of Q / K tile
    static constexpr uint32_t Q_BYTES = kRows * D * 2;
    static constexpr uint32_t KV_BYTES = BN * D * 2;          // one K (or V) block
    static constexpr int NO = (2 * BN + 2 * D <= int(kTmemCols)) ? 2 : 1;   // O buffers in TMEM
    static constexpr int NQ = (2 * Q_BYTES + 4 * KV_BYTES <= 200u * 1024u) ? 2 : 1;   // Q buffers in smem
    static constexpr uint32_t OFF_Q = 0;                      // [NQ] Q buffers
    static constexpr uint32_t OFF_K = OFF_Q + NQ * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr uint32_t OFF_X = OFF_V + STAGES * KV_BYTES;   // [2 parity][2 wg][128] max exchange
    static constexpr uint32_t OFF_LX = OFF_X + 2 * 2 * kRows * 4;    // [128] l exchange
    static constexpr uint32_t OFF_BAR = OFF_LX + kRows * 4;
    static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;    // + barriers, + alignment slack
    // TMEM columns: S buffers at 0 and BN (P overwrites each half's first
    // quarter), O buffers after them.
    static constexpr uint32_t COL_S = 0, COL_O = 2 * BN;
    static_assert(2 * BN + NO * D <= int(kTmemCols), "TMEM budget");
    static_assert(SMEM <= 227 * 1024, "shared memory budget");
};

struct TcParams {
    AttnParams a;
    int nsplit;
    int split_keys;     // keys per split (multiple of BN)
    int n_items;
};

enum : int {
    B_KFULL = 0,    // [2]
    B_KEMPTY = 2,   // [2]
    B_VFULL = 4,    // [2]
    B_VEMPTY = 6,   // [2]
    B_SFULL = 8,    // [2] S block computed
    B_SFREE = 10,   // [2] P of the block consumed by P V (S buffer reusable, O updated)
    B_PFULL = 12,   // [2] P written (and O rescaled) by the softmax threads
    B_QFULL = 14,   // [2]
    B_QEMPTY = 16,  // [2]
    B_ODONE = 18,   // [2]
    B_OFREE = 20,   // [2]
    B_DRAIN = 22,
    B_XCH = 23,     // [2] block-maximum exchange between the two softmax halves
    B_LXCH = 25,    // row-sum exchange at an item's end
    B_COUNT = 26
};

// Decode work item -> tile, kv head, split (consecutive items = consecutive
// tiles of one (head, split), so a group's tiles read its span together).
struct ItemInfo {
    int tile, h, split, grp, first, nseq, k0, k1, nblk;
    long span_row;      // first row of the span in the store's 2D view
    bool donor;
};

template <int D>
__device__ __forceinline__ ItemInfo item_info(const AttnParams& P, const TcParams& tp, int item) {
    ItemInfo it;
    it.tile = item % P.n_tiles;
    const int hs = item / P.n_tiles;
    it.split = hs % tp.nsplit;
    it.h = hs / tp.nsplit;
    const int4 tl = reinterpret_cast<const int4*>(P.tiles)[it.tile];
    it.grp = tl.x;
    it.first = tl.y;
    it.nseq = tl.z;
    const int prompt = P.group_prompt[it.grp];
    const int code = P.group_src[it.grp];
    it.donor = code != int(SPLICE_SRC_CLEAN);
    long span;
    if (!it.donor) {
        span = (long(prompt) * P.N + P.layer) * P.Hkv + it.h;
    } else {
        const int st = P.slot_stored[code - int(SPLICE_SRC_DONOR0)];
        span = ((long(prompt) * P.Dst + st) * P.N + P.layer) * P.Hkv + it.h;
    }
    it.span_row = span * P.Tp;
    it.k0 = P.p_lo + it.split * tp.split_keys;
    it.k1 = min(P.p_hi, it.k0 + tp.split_keys);
    it.nblk = it.k1 > it.k0 ? (it.k1 - it.k0 + Cfg<D>::BN - 1) / Cfg<D>::BN : 0;
    return it;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_tc_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                     const __grid_constant__ CUtensorMap tm_kd, const __grid_constant__ CUtensorMap tm_vd,
                     const TcParams tp) {
    using C = Cfg<D>;
    const AttnParams& P = tp.a;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = tc::smem_u32(smem);
    const uint32_t bar0 = sbase + C::OFF_BAR;
    auto bar = [&](int i) { return bar0 + 8u * uint32_t(i); };
    volatile int* s_abort = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 8 * B_COUNT);
    uint32_t* s_tmem = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 8 * B_COUNT + 8);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(bar(B_KFULL + i), 1);
            tc::mbar_init(bar(B_KEMPTY + i), 1);
            tc::mbar_init(bar(B_VFULL + i), 1);
            tc::mbar_init(bar(B_VEMPTY + i), 1);
            tc::mbar_init(bar(B_SFULL + i), 1);
            tc::mbar_init(bar(B_SFREE + i), 1);
            tc::mbar_init(bar(B_PFULL + i), kSoftmaxThreads);
            tc::mbar_init(bar(B_QFULL + i), 32);
            tc::mbar_init(bar(B_QEMPTY + i), 1);
            tc::mbar_init(bar(B_ODONE + i), 1);
            tc::mbar_init(bar(B_OFREE + i), kSoftmaxThreads);
        }
        tc::mbar_init(bar(B_DRAIN), 1);
        tc::mbar_init(bar(B_XCH), kSoftmaxThreads);
        tc::mbar_init(bar(B_XCH + 1), kSoftmaxThreads);
        tc::mbar_init(bar(B_LXCH), kSoftmaxThreads);
        *s_abort = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(&tm_kc);
        tc::prefetch_tmap(&tm_vc);
        tc::prefetch_tmap(&tm_kd);
        tc::prefetch_tmap(&tm_vd);
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(s_tmem), kTmemCols);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *s_tmem;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int jg = 0;          // global block counter of this CTA
            int issued_k = 0, issued_v = 0;
            for (int item = blockIdx.x; item < tp.n_items && !*s_abort; item += gridDim.x) {
                const ItemInfo it = item_info<D>(P, tp, item);
                const CUtensorMap* tmk = it.donor ? &tm_kd : &tm_kc;
                const CUtensorMap* tmv = it.donor ? &tm_vd : &tm_vc;
                for (int j = 0; j < it.nblk && !*s_abort; ++j, ++jg) {
                    const int stg = jg % C::STAGES;
                    const uint32_t use = uint32_t(jg / C::STAGES);
                    const int y = int(it.span_row + it.k0 + j * C::BN);
                    if (!tc::mbar_wait(bar(B_KEMPTY + stg), (use & 1u) ^ 1u, s_abort, P.err, kErrWaitProducer)) break;
                    tc::mbar_arrive_expect_tx(bar(B_KFULL + stg), C::KV_BYTES);
#pragma unroll
                    for (int b = 0; b < C::KB; ++b)
                        tc::tma_load_2d(sbase + C::OFF_K + stg * C::KV_BYTES + b * (C::BN * 128), tmk, b * 64, y,
                                        bar(B_KFULL + stg));
                    issued_k = jg + 1;
                    if (!tc::mbar_wait(bar(B_VEMPTY + stg), (use & 1u) ^ 1u, s_abort, P.err, kErrWaitProducer)) break;
                    tc::mbar_arrive_expect_tx(bar(B_VFULL + stg), C::KV_BYTES);
#pragma unroll
                    for (int b = 0; b < C::KB; ++b)
                        tc::tma_load_2d(sbase + C::OFF_V + stg * C::KV_BYTES + b * (C::BN * 128), tmv, b * 64, y,
                                        bar(B_VFULL + stg));
                    issued_v = jg + 1;
                }
            }
            // Drain: every issued copy must land before the CTA may exit.
            for (int j = max(0, issued_k - C::STAGES); j < issued_k; ++j) {
                volatile int no_abort = 0;
                tc::mbar_wait(bar(B_KFULL + j % C::STAGES), uint32_t(j / C::STAGES) & 1u, &no_abort, P.err,
                              kErrWaitDrain);
            }
            for (int j = max(0, issued_v - C::STAGES); j < issued_v; ++j) {
                volatile int no_abort = 0;
                tc::mbar_wait(bar(B_VFULL + j % C::STAGES), uint32_t(j / C::STAGES) & 1u, &no_abort, P.err,
                              kErrWaitDrain);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_qk = tc::idesc_bf16_f32(kRows, C::BN, false);
            constexpr uint32_t idesc_pv = tc::idesc_bf16_f32(kRows, D, true);
            bool ok = true, committed = false;
            int jg = 0, n_item = 0;
            for (int item = blockIdx.x; ok && item < tp.n_items; item += gridDim.x, ++n_item) {
                const ItemInfo it = item_info<D>(P, tp, item);
                const int qb = C::NQ == 2 ? (n_item & 1) : 0;
                const uint32_t quse = uint32_t(C::NQ == 2 ? n_item >> 1 : n_item);
                const int ob = C::NO == 2 ? (n_item & 1) : 0;
                const uint32_t ouse = uint32_t(C::NO == 2 ? n_item >> 1 : n_item);
                const uint32_t q_addr = sbase + C::OFF_Q + qb * C::Q_BYTES;
                const uint32_t o_col = tmem + C::COL_O + ob * D;
                if (!tc::mbar_wait(bar(B_QFULL + qb), quse & 1u, s_abort, P.err, kErrWaitMma)) {
                    ok = false;
                    break;
                }
                auto pv = [&](int jgp, int jl) -> bool {
                    const int stg = jgp % C::STAGES;
                    const int sb = jgp & 1;
                    if (!tc::mbar_wait(bar(B_PFULL + sb), uint32_t(jgp >> 1) & 1u, s_abort, P.err, kErrWaitMma))
                        return false;
                    if (!tc::mbar_wait(bar(B_VFULL + stg), uint32_t(jgp / C::STAGES) & 1u, s_abort, P.err,
                                       kErrWaitMma))
                        return false;
                    if (jl == 0 &&
                        !tc::mbar_wait(bar(B_OFREE + ob), (ouse & 1u) ^ 1u, s_abort, P.err, kErrWaitMma))
                        return false;
                    tc::tc_fence_after();
                    const uint32_t v_addr = sbase + C::OFF_V + stg * C::KV_BYTES;
                    const uint32_t p_col = tmem + C::COL_S + sb * C::BN;
#pragma unroll
                    for (int kk = 0; kk < C::BN / 16; ++kk) {
                        // 16 keys of P: two bf16 per TMEM column; the first
                        // half's P sits at the start of its S half, the second
                        // half's at the start of the other S half.
                        const int half = kk / (C::HALF / 16);
                        const int kin = kk % (C::HALF / 16);
                        const uint32_t a = p_col + half * C::HALF + kin * 8;
                        const uint64_t b = tc::sw128_desc(v_addr + kk * 16 * 128, C::BN * 128, 1024);
                        mma_f16_ts(o_col, a, b, idesc_pv, (jl > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(bar(B_SFREE + sb));
                    tc::mma_commit(bar(B_VEMPTY + stg));
                    committed = true;
                    return true;
                };
                for (int j = 0; j < it.nblk; ++j, ++jg) {
                    const int stg = jg % C::STAGES;
                    const int sb = jg & 1;
                    if (!tc::mbar_wait(bar(B_KFULL + stg), uint32_t(jg / C::STAGES) & 1u, s_abort, P.err, kErrWaitMma) ||
                        !tc::mbar_wait(bar(B_SFREE + sb), (uint32_t(jg >> 1) & 1u) ^ 1u, s_abort, P.err, kErrWaitMma)) {
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
                    const uint32_t k_addr = sbase + C::OFF_K + stg * C::KV_BYTES;
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint64_t a = tc::sw128_desc(q_addr + (kk / 4) * (kRows * 128) + (kk % 4) * 32, 16, 1024);
                        const uint64_t b = tc::sw128_desc(k_addr + (kk / 4) * (C::BN * 128) + (kk % 4) * 32, 16, 1024);
                        tc::mma_f16_ss(tmem + C::COL_S + sb * C::BN, a, b, idesc_qk, kk > 0 ? 1u : 0u);
                    }
                    tc::mma_commit(bar(B_SFULL + sb));
                    tc::mma_commit(bar(B_KEMPTY + stg));
                    if (j == it.nblk - 1) tc::mma_commit(bar(B_QEMPTY + qb));
                    committed = true;
                    if (j >= 1 && !pv(jg - 1, j - 1)) {
                        ok = false;
                        break;
                    }
                }
                if (!ok) break;
                if (it.nblk > 0) {
                    if (!pv(jg - 1, it.nblk - 1)) {
                        ok = false;
                        break;
                    }
                } else {
                    tc::mma_commit(bar(B_QEMPTY + qb));
                }
                tc::mma_commit(bar(B_ODONE + ob));
            }
            if (!ok && committed) {
                // Let the MMAs already issued finish before TMEM is freed.
                tc::mma_commit(bar(B_DRAIN));
                volatile int no_abort = 0;
                tc::mbar_wait(bar(B_DRAIN), 0, &no_abort, P.err, kErrWaitDrain);
            }
        }
    } else if (warp == 2) {
        // ------------------------------------------------ Q gather
        int n_item = 0;
        for (int item = blockIdx.x; item < tp.n_items; item += gridDim.x, ++n_item) {
            const ItemInfo it = item_info<D>(P, tp, item);
            const int qb = C::NQ == 2 ? (n_item & 1) : 0;
            const uint32_t quse = uint32_t(C::NQ == 2 ? n_item >> 1 : n_item);
            const bool got = tc::mbar_wait(bar(B_QEMPTY + qb), (quse & 1u) ^ 1u, s_abort, P.err, kErrWaitQ);
            if (!__all_sync(0xffffffffu, got)) break;
            uint8_t* q_s = smem + C::OFF_Q + qb * C::Q_BYTES;
            const int nrows = it.nseq * P.G;
#pragma unroll 1
            for (int rr = 0; rr < kRows / 32; ++rr) {
                const int row = rr * 32 + lane;
                uint4 v[D / 8];
                if (row < nrows) {
                    const int s = P.group_seqs[it.first + row / P.G];
                    const int hq = it.h * P.G + row % P.G;
                    const uint4* src = reinterpret_cast<const uint4*>(P.q + (long(s) * P.Hq + hq) * D);
#pragma unroll
                    for (int c = 0; c < D / 8; ++c) v[c] = src[c];
                } else {
#pragma unroll
                    for (int c = 0; c < D / 8; ++c) v[c] = make_uint4(0, 0, 0, 0);
                }
#pragma unroll
                for (int c = 0; c < D / 8; ++c)
                    *reinterpret_cast<uint4*>(q_s + (c / 8) * (kRows * 128) + row * 128 + (((c % 8) ^ (row % 8)) * 16)) =
                        v[c];
            }
            tc::fence_proxy_async_smem();
            tc::mbar_arrive(bar(B_QFULL + qb));
        }
    } else {
        // ------------------------------------------------ softmax / epilogue
        const int wg = (warp - 3) / 4;                 // 0: first half of each block's keys, 1: second half
        const int quarter = warp & 3;                  // TMEM lane quarter this warp may access
        const int row = quarter * 32 + lane;           // == TMEM lane of this thread's row
        const uint32_t lane_base = uint32_t(quarter * 32) << 16;
        float* xmax = reinterpret_cast<float*>(smem + C::OFF_X);
        float* xl = reinterpret_cast<float*>(smem + C::OFF_LX);
        const float c = P.scale_log2;
        bool ok = true;
        int jg = 0, n_item = 0, n_lx = 0;
        for (int item = blockIdx.x; ok && item < tp.n_items; item += gridDim.x, ++n_item) {
            const ItemInfo it = item_info<D>(P, tp, item);
            const int ob = C::NO == 2 ? (n_item & 1) : 0;
            const uint32_t ouse = uint32_t(C::NO == 2 ? n_item >> 1 : n_item);
            const bool valid = row < it.nseq * P.G;
            long out_row = 0;
            if (valid) {
                const int s = P.group_seqs[it.first + row / P.G];
                out_row = long(s) * P.Hq + it.h * P.G + row % P.G;
            }
            float m_run = -INFINITY, l_run = 0.f;
            for (int j = 0; j < it.nblk; ++j, ++jg) {
                const int sb = jg & 1;
                // waits are made warp-uniform: tcgen05.ld/st are warp-collective
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_SFULL + sb), uint32_t(jg >> 1) & 1u, s_abort, P.err,
                                                           kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t s_col = tmem + lane_base + C::COL_S + sb * C::BN + wg * C::HALF;
                float s[C::HALF];
#pragma unroll
                for (int q = 0; q < C::HALF / 32; ++q) {
                    float v[32];
                    tc::tmem_ld32(s_col + q * 32, v);
#pragma unroll
                    for (int i = 0; i < 32; ++i) s[q * 32 + i] = v[i];
                }
                tc::tmem_wait_ld();
                // keys past the split end are masked (only the last block)
                const int kbase = it.k0 + j * C::BN + wg * C::HALF;
                const bool tail = kbase + C::HALF > it.k1;
                if (tail) {
#pragma unroll
                    for (int i = 0; i < C::HALF; ++i)
                        if (kbase + i >= it.k1) s[i] = c >= 0.f ? -INFINITY : INFINITY;
                }
                // block extreme of the raw logits in this half (max for c >= 0)
                float e0 = s[0], e1 = s[1], e2 = s[2], e3 = s[3];
                if (c >= 0.f) {
#pragma unroll
                    for (int i = 4; i < C::HALF; i += 4) {
                        e0 = fmaxf(e0, s[i]);
                        e1 = fmaxf(e1, s[i + 1]);
                        e2 = fmaxf(e2, s[i + 2]);
                        e3 = fmaxf(e3, s[i + 3]);
                    }
                    e0 = fmaxf(fmaxf(e0, e1), fmaxf(e2, e3));
                } else {
#pragma unroll
                    for (int i = 4; i < C::HALF; i += 4) {
                        e0 = fminf(e0, s[i]);
                        e1 = fminf(e1, s[i + 1]);
                        e2 = fminf(e2, s[i + 2]);
                        e3 = fminf(e3, s[i + 3]);
                    }
                    e0 = fminf(fminf(e0, e1), fminf(e2, e3));
                }
                float* xm = xmax + (jg & 1) * (2 * kRows);
                xm[wg * kRows + row] = e0;
                tc::mbar_arrive(bar(B_XCH + (jg & 1)));
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_XCH + (jg & 1)), uint32_t(jg >> 1) & 1u, s_abort,
                                                           P.err, kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                const float eo = xm[(wg ^ 1) * kRows + row];
                const float ext = c >= 0.f ? fmaxf(e0, eo) : fminf(e0, eo);
                const float mc = ext * c;                      // block max in log2 units
                float alpha = 1.f;
                bool resc = false;
                if (mc > m_run + kTau) {
                    alpha = ex2(m_run - mc);
                    resc = j > 0;
                    m_run = mc;
                }
                const float nm = -m_run;
                float lsum = 0.f;
                uint32_t pk[C::HALF / 2];
#pragma unroll
                for (int i = 0; i < C::HALF / 2; ++i) {
                    float a = ex2(fmaf(s[2 * i], c, nm));
                    float b = ex2(fmaf(s[2 * i + 1], c, nm));
                    if (tail) {
                        a = kbase + 2 * i < it.k1 ? a : 0.f;
                        b = kbase + 2 * i + 1 < it.k1 ? b : 0.f;
                    }
                    lsum += a + b;
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(a, b);
                    pk[i] = *reinterpret_cast<const uint32_t*>(&h2);
                }
                if (__any_sync(0xffffffffu, resc)) {
                    // O must hold P V of every earlier block of this item
                    if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_SFREE + ((jg - 1) & 1)),
                                                               uint32_t((jg - 1) >> 1) & 1u, s_abort, P.err,
                                                               kErrWaitSoftmax))) {
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
#pragma unroll
                    for (int q = 0; q < D / 64; ++q) {
                        float v[32];
                        const uint32_t ta = tmem + lane_base + C::COL_O + ob * D + wg * (D / 2) + q * 32;
                        tc::tmem_ld32(ta, v);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= resc ? alpha : 1.f;
                        tc::tmem_st32(ta, v);
                    }
                    tc::tmem_wait_st();
                }
                l_run = l_run * alpha + lsum;
                // P (bf16 pairs) over the first quarter of this half's S columns
                const uint32_t p_col = tmem + lane_base + C::COL_S + sb * C::BN + wg * C::HALF;
                if constexpr (C::HALF / 2 == 32) {
                    uint32_t lo[16], hi[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        lo[i] = pk[i];
                        hi[i] = pk[16 + i];
                    }
                    tmem_st16(p_col, lo);
                    tmem_st16(p_col + 16, hi);
                } else {
                    tmem_st16(p_col, *reinterpret_cast<const uint32_t(*)[16]>(pk));
                }
                tc::tmem_wait_st();
                tc::tc_fence_before();
                tc::mbar_arrive(bar(B_PFULL + sb));
            }
            if (!ok) break;
            // ---- epilogue: partial state of this row for this item ----
            if (it.nblk > 0) {
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_ODONE + ob), ouse & 1u, s_abort, P.err,
                                                           kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const size_t idx = size_t(it.split) * P.B * P.Hq + size_t(out_row);
                float* op = P.ws_o + idx * D + wg * (D / 2);
#pragma unroll
                for (int q = 0; q < D / 64; ++q) {
                    float v[32];
                    tc::tmem_ld32(tmem + lane_base + C::COL_O + ob * D + wg * (D / 2) + q * 32, v);
                    tc::tmem_wait_ld();
                    if (valid) {
#pragma unroll
                        for (int i = 0; i < 32; i += 4)
                            *reinterpret_cast<float4*>(op + q * 32 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                    }
                }
                if (wg == 1) xl[row] = l_run;
                tc::mbar_arrive(bar(B_LXCH));
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_LXCH), uint32_t(n_lx) & 1u, s_abort, P.err,
                                                           kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                ++n_lx;
                if (wg == 0 && valid) P.ws_ml[idx] = make_float2(m_run, l_run + xl[row]);
                tc::tc_fence_before();
                tc::mbar_arrive(bar(B_OFREE + ob));
            } else {
                // an empty split: a state with no keys
                if (wg == 0 && valid) {
                    const size_t idx = size_t(it.split) * P.B * P.Hq + size_t(out_row);
                    P.ws_ml[idx] = make_float2(-INFINITY, 0.f);
                }
                tc::mbar_arrive(bar(B_OFREE + ob));
                // matching the MMA side: it commits ODONE for an empty item too
                tc::mbar_wait(bar(B_ODONE + ob), ouse & 1u, s_abort, P.err, kErrWaitSoftmax);
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (warp == 1) tc::tmem_dealloc(tmem, kTmemCols);
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no -lcuda).
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
    static EncodeFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeFn>(p);
    }
    return fn;
}

template <int D>
void launch_d(const TcParams& tp, const CUtensorMap* m, cudaStream_t st) {
    static int sms = 0;
    if (!sms) {
        cudaFuncSetAttribute(prefix_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<D>::SMEM);
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    const unsigned grid = unsigned(tp.n_items < sms ? tp.n_items : sms);
    prefix_tc_kernel<D><<<grid, kThreads, Cfg<D>::SMEM, st>>>(m[0], m[1], m[2], m[3], tp);
}

}  // namespace

// 2D view [rows][d] of a bf16 store; box = 64 elements x box_rows rows, 128-byte swizzle.
int make_kv_tensor_map(void* out_map, const void* base, long rows, int d, int box_rows) {
    EncodeFn enc = encode_fn();
    if (!enc) return int(cudaErrorNotSupported);
    if (rows < 1) rows = 1;
    const cuuint64_t dims[2] = {cuuint64_t(d), cuuint64_t(rows)};
    const cuuint64_t strides[1] = {cuuint64_t(d) * 2};
    const cuuint32_t box[2] = {64, cuuint32_t(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(static_cast<CUtensorMap*>(out_map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
                     dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? 0 : int(cudaErrorInvalidValue);
}

int prefix_tc_box_rows(int d) { return d == 256 ? Cfg<256>::BN : 128; }

int prefix_tc_split_keys(int d, int p_vis, int* nsplit) {
    const int bn = prefix_tc_box_rows(d);
    // Splits depend only on the visible span length, so a row's arithmetic
    // never depends on which other rows share its tile or launch.
    int ns = (p_vis + 1023) / 1024;
    ns = ns < 1 ? 1 : (ns > kMaxPrefixSplits ? kMaxPrefixSplits : ns);
    int keys = (p_vis + ns - 1) / ns;
    keys = (keys + bn - 1) / bn * bn;
    ns = (p_vis + keys - 1) / keys;
    *nsplit = ns;
    return keys;
}

int launch_prefix_tc(const AttnParams& p, const void* maps, int nsplit, int split_keys, void* stream) {
    const CUtensorMap* m = static_cast<const CUtensorMap*>(maps);
    TcParams tp{p, nsplit, split_keys, p.n_tiles * p.Hkv * nsplit};
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.D) {
        case 64: launch_d<64>(tp, m, st); break;
        case 128: launch_d<128>(tp, m, st); break;
        case 256: launch_d<256>(tp, m, st); break;
        default: return int(cudaErrorInvalidValue);
    }
    return int(cudaGetLastError());
}

}  // namespace splice
