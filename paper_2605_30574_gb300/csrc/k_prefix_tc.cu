// Tensor-core prompt-span pass (tcgen05 + TMEM, TMA-fed), persistent.
//
// Every sequence that reads the same (prompt, source) span at a (layer,
// step) -- a group of the descriptor's table -- shares that span's K/V.  For
// one kv head h, the G query rows of every sequence of the group are stacked
// into 128-row tiles, so Q K^T and P V over the span are dense contractions
// (M = 128 stacked rows).  A work item is one (row tile, kv head, key
// split).  Items are handed out at run time: each CTA's producer claims the
// next item from a launch-wide counter and posts it to the CTA's other roles
// through a small ring in smem, so CTAs that draw short items take more.
//
//   warp 0        TMA producer (one lane, two cursors): claims items; K and V
//                 blocks of the item's span -> two-stage smem rings, each
//                 block loaded as soon as its stage is free
//   warp 1        Q K^T issuer (one elected lane): S of the next key block
//                 into a free TMEM slot (NSLOT slots); owns the TMEM
//                 allocation
//   warp 2        Q gather: the tile's query rows -> smem with cp.async,
//                 one item ahead
//   warps 4..11   softmax, two warpgroups: each thread owns one row and one
//                 half of every block's keys; the halves trade block maxima
//                 through smem, share one lazily moved reference max, write
//                 P (bf16) over their own half of the slot in TMEM, rescale
//                 their half of O when the reference moves, and at the item's
//                 end write the row's partial state (m, l, o) to the
//                 workspace, through a per-warp staging buffer so the stores
//                 leave in row-contiguous pieces.  Warps whose 32 rows are all past the tile's end
//                 skip the arithmetic but keep every barrier.
//   warp 3        P V issuer (one elected lane): O += P V with P read from
//                 TMEM as soon as the softmax has written it -- a separate
//                 issuer, so P V never queues behind the next Q K^T
//
// Delta mode: a tile of a clean span may hold rows of readers of a
// delta-encoded donor; for those rows the softmax drops the slot's encoded
// positions (a per-row bitmask), and items over the slot's encoded rows (a
// store of their own, split like a span) give the rest of the donor span.
//
// The merge kernel (or, with this pass first and one split of each span, the
// generated-span pass) combines these partials with those of the generated
// span (and the ZERO closed form).  Every wait is bounded: a wait that runs out
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

constexpr int kRows = 128;          // MMA M, rows of one tile
constexpr int kWarps = 12;          // producer, Q K^T issuer, Q gather, P V issuer, 8 softmax
constexpr int kPvWarp = 3;
// Register split (setmaxnreg, per warpgroup): warps 0-3 give registers to
// the two softmax warpgroups.  256 * 184 + 128 * 112 = 61440 <= the launch's
// 384 threads * 168.
constexpr uint32_t kRegsControl = 112, kRegsSoftmax = 184;
constexpr int kThreads = kWarps * 32;
constexpr uint32_t kTmemCols = 512;
constexpr float kTau = 8.0f;        // lazy rescale threshold, log2 units

constexpr unsigned kErrWaitProducer = 0x1, kErrWaitMma = 0x2, kErrWaitSoftmax = 0x4, kErrWaitDrain = 0x8,
                   kErrWaitQ = 0x20, kErrWaitItem = 0x40;
// Work items reach the CTA's roles through a ring in smem: the producer
// posts every item decoded (tile, kv head, split, span), so no other role
// reads the tile tables.
constexpr int kItemRing = 8;
constexpr int kItemTakers = 12;     // Q K^T warp, P V warp, Q gather warp, 8 softmax warps, the V cursor
constexpr uint32_t kRingEntryBytes = 64;

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

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&v)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr),
                 "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
                 : "memory");
}

// One segment's P (bf16 pairs), by segment size.
__device__ __forceinline__ void store_p(uint32_t taddr, const uint32_t (&v)[16]) { tmem_st16(taddr, v); }
__device__ __forceinline__ void store_p(uint32_t taddr, const uint32_t (&v)[8]) { tmem_st8(taddr, v); }

// SHORT: every item of the launch has at most four key blocks (prompt spans
// of up to 512 keys at d <= 128).  A V block then waits only briefly for its
// P V, so V takes the two-stage ring of K and the smem goes to a second Q
// buffer: the next item's queries are gathered while this item runs, instead
// of after its last Q K^T.
template <int D, bool SHORT = false>
struct Cfg {
    static constexpr int BN = D == 256 ? 64 : 128;          // keys per K/V block
    static constexpr int KPT = BN / 2;                      // keys per softmax thread per block
    static constexpr int OCH = D / 2;                       // O columns per softmax thread
    static constexpr int KB = D / 64;                       // 64-wide column blocks of Q / K / V
    static constexpr uint32_t KV_BYTES = BN * D * 2;        // one K (or V) block
    // A V block stays in smem from its load until its P V has run, several
    // blocks later, so V gets the deeper ring: 192 KB of Q, K and V stages.
    static constexpr uint32_t Q_BYTES = kRows * D * 2;      // Q of one tile
    static constexpr int KST = int((64u * 1024u) / KV_BYTES);      // K stages: 64 KB
    static constexpr int VST = (D == 256 || SHORT) ? KST : KST + KST / 2;   // V stages: 96 KB where smem allows
    static constexpr int NQ = (2 * Q_BYTES + (KST + VST) * KV_BYTES <= 192u * 1024u) ? 2 : 1;   // Q buffers
    // TMEM columns: NSLOT slots of BN columns for S (each softmax thread's
    // P over the first columns of its half of the slot), then O.
    static constexpr int NSLOT = (int(kTmemCols) - D) / BN > 4 ? 4 : (int(kTmemCols) - D) / BN;
    static constexpr uint32_t COL_O = NSLOT * BN;
    static constexpr uint32_t OFF_Q = 0;                    // [NQ] Q buffers
    static constexpr uint32_t OFF_K = OFF_Q + NQ * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + KST * KV_BYTES;
    // exchange: [2 parity][2 half][128] block maxima, [2 parity][2 half][128] row sums
    static constexpr uint32_t OFF_X = OFF_V + VST * KV_BYTES;
    static constexpr uint32_t X_BYTES = 2 * (2 * 2 * kRows) * 4;
    static constexpr uint32_t OFF_BAR = OFF_X + X_BYTES;
    static constexpr uint32_t OFF_RING = OFF_BAR + 1024;    // [kItemRing] posted work items
    // [8 softmax warps][32 rows][16 floats]: the epilogue's staging, so the
    // partial states leave in row-contiguous 64-byte pieces
    static constexpr uint32_t OFF_STG = (OFF_RING + kItemRing * kRingEntryBytes + 127) / 128 * 128;
    static constexpr uint32_t STG_BYTES = 32 * 16 * 4;
    static constexpr uint32_t SMEM = OFF_STG + 8 * STG_BYTES + 1024;   // + alignment slack
    static_assert(NSLOT >= 2 && COL_O + D <= kTmemCols, "TMEM budget");
    static_assert(SMEM <= 227 * 1024, "shared memory budget");
    static_assert(KPT % 32 == 0 && OCH % 32 == 0 && VST >= 2, "TMEM access granularity, ring depth");
};

// Barrier indices (8 bytes each from OFF_BAR).
template <int KST, int VST, int NSLOT>
struct Bars {
    static constexpr int KFULL = 0;                       // [KST]
    static constexpr int KEMPTY = KST;                    // [KST]
    static constexpr int VFULL = 2 * KST;                 // [VST]
    static constexpr int VEMPTY = 2 * KST + VST;          // [VST]
    static constexpr int SFULL = 2 * KST + 2 * VST;       // [NSLOT] S computed
    static constexpr int SFREE = SFULL + NSLOT;           // [NSLOT] P of the slot consumed by P V
    static constexpr int PFULL = SFREE + NSLOT;           // [NSLOT] P written (and O rescaled)
    static constexpr int QFULL = PFULL + NSLOT;           // [2]
    static constexpr int QEMPTY = QFULL + 2;              // [2]
    static constexpr int ODONE = QEMPTY + 2;
    static constexpr int OFREE = ODONE + 1;
    static constexpr int DRAIN = OFREE + 1;               // [issuer]
    static constexpr int XCH = DRAIN + 2;                 // [2 parity][4 lane quarters] block-maximum exchange
    static constexpr int LXCH = XCH + 8;                  // row-sum exchange at an item's end
    static constexpr int IFULL = LXCH + 1;                // [kItemRing] item number posted
    static constexpr int IEMPTY = IFULL + kItemRing;      // [kItemRing] item number taken by every role
    static constexpr int COUNT = IEMPTY + kItemRing;
    static_assert(COUNT * 8 + 16 + 4 * kItemRing <= 1024, "barrier area");
};

struct TcParams {
    AttnParams a;
    int sb[kMaxPrefixSplits + 1];   // split boundaries of a stored span, relative to p_lo (multiples of BN)
    int delta_keys;                 // keys per split of the delta rows (multiple of BN)
    int n_span_items;               // items [0, n_span_items) read stored spans, the rest delta rows
    int n_items;
};

// Work item -> tile, kv head, split (consecutive items = consecutive tiles
// of one (head, split), so a group's tiles read its span at about the same
// time and share it in L2; split-major, so the run-time queue hands out the
// first -- longest -- split of every span before the shorter ones and the
// launch ends on short items).  Items over stored spans come first, then
// the items over delta rows (their own split count).
struct ItemInfo {
    int item;           // the item's number; -1 after the CTA's last item, -2 when a wait gave up
    int h, split, first, nseq, k0, k1, nblk, prompt;
    int store;          // 0 clean, 1 donor, 2 delta rows
    bool masked;        // a clean span in delta mode: rows may drop encoded positions
    long span_row;      // first row of the span in the store's 2D view
};
static_assert(sizeof(ItemInfo) <= kRingEntryBytes, "item ring entry");

template <int D>
__device__ __forceinline__ ItemInfo item_info(const AttnParams& P, const TcParams& tp, int item) {
    ItemInfo it;
    it.item = item;
    int tile, split;
    if (item < tp.n_span_items) {
        tile = item % P.n_span_tiles;
        const int hs = item / P.n_span_tiles;
        it.h = hs % P.Hkv;
        split = hs / P.Hkv;
        it.split = split;                      // partial slot
    } else {
        const int nd = P.n_tiles - P.n_span_tiles;
        const int j = item - tp.n_span_items;
        tile = P.n_span_tiles + j % nd;
        const int hs = j / nd;
        it.h = hs % P.Hkv;
        split = hs / P.Hkv;
        it.split = P.nsp + split;              // after the span's own partials
    }
    // one 16-byte record per tile: group, first reader, readers, and the
    // store kind with the span base index (clean: the prompt; donor or delta
    // rows: prompt * stored slots + stored index)
    const int4 tl = reinterpret_cast<const int4*>(P.tiles)[tile];
    it.first = tl.y;
    it.nseq = tl.z;
    it.store = tl.w & 3;
    const long base = long(unsigned(tl.w) >> 2);
    it.prompt = int(base);                     // used by clean spans only
    const long span = (base * P.N + P.layer) * P.Hkv + it.h;
    if (it.store == 2) {
        it.masked = false;
        it.k0 = split * tp.delta_keys;
        it.k1 = min(P.dcount[span], it.k0 + tp.delta_keys);
    } else {
        it.masked = it.store == 0 && P.delta_on != 0;
        it.k0 = P.p_lo + tp.sb[split];
        it.k1 = P.p_lo + tp.sb[split + 1];
    }
    it.span_row = span * P.Tp;
    it.nblk = it.k1 > it.k0 ? (it.k1 - it.k0 + Cfg<D>::BN - 1) / Cfg<D>::BN : 0;
    return it;
}

template <int D, bool SHORT>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_tc_kernel(const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
                     const __grid_constant__ CUtensorMap tm_kd, const __grid_constant__ CUtensorMap tm_vd,
                     const __grid_constant__ CUtensorMap tm_kx, const __grid_constant__ CUtensorMap tm_vx,
                     const TcParams tp) {
    using C = Cfg<D, SHORT>;
    using Bb = Bars<C::KST, C::VST, C::NSLOT>;
    constexpr int NSLOT = C::NSLOT;
    const AttnParams& P = tp.a;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = tc::smem_u32(smem);
    const uint32_t bar0 = sbase + C::OFF_BAR;
    auto bar = [&](int i) { return bar0 + 8u * uint32_t(i); };
    volatile int* s_abort = reinterpret_cast<volatile int*>(smem + C::OFF_BAR + 8 * Bb::COUNT);
    uint32_t* s_tmem = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + 8 * Bb::COUNT + 8);
    // The producer posts every item with its decoded fields, so no other
    // role reads the tile tables.
    ItemInfo* s_ring = reinterpret_cast<ItemInfo*>(smem + C::OFF_RING);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::KST; ++i) {
            tc::mbar_init(bar(Bb::KFULL + i), 1);
            tc::mbar_init(bar(Bb::KEMPTY + i), 1);
        }
        for (int i = 0; i < C::VST; ++i) {
            tc::mbar_init(bar(Bb::VFULL + i), 1);
            tc::mbar_init(bar(Bb::VEMPTY + i), 1);
        }
        for (int i = 0; i < NSLOT; ++i) {
            tc::mbar_init(bar(Bb::SFULL + i), 1);
            tc::mbar_init(bar(Bb::SFREE + i), 1);
            tc::mbar_init(bar(Bb::PFULL + i), 256);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(bar(Bb::QFULL + i), 32);
            tc::mbar_init(bar(Bb::QEMPTY + i), 1);
            for (int q = 0; q < 4; ++q) tc::mbar_init(bar(Bb::XCH + 4 * i + q), 64);   // the quarter's two warps
            tc::mbar_init(bar(Bb::DRAIN + i), 1);
        }
        tc::mbar_init(bar(Bb::ODONE), 1);
        tc::mbar_init(bar(Bb::OFREE), 256);
        tc::mbar_init(bar(Bb::LXCH), 256);
        for (int i = 0; i < kItemRing; ++i) {
            tc::mbar_init(bar(Bb::IFULL + i), 1);
            tc::mbar_init(bar(Bb::IEMPTY + i), kItemTakers);
        }
        *s_abort = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(&tm_kc);
        tc::prefetch_tmap(&tm_vc);
        tc::prefetch_tmap(&tm_kd);
        tc::prefetch_tmap(&tm_vd);
        if (P.delta_on) {
            tc::prefetch_tmap(&tm_kx);
            tc::prefetch_tmap(&tm_vx);
        }
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(s_tmem), kTmemCols);
        tc::tmem_relinquish();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    // The call's first pass: launched as a programmatic dependent of
    // whatever precedes it on the stream, this grid may start before that
    // work has finished, so it waits for it (its writes visible) before
    // reading anything -- the queries, the work counter, the tables.  Only
    // then may the generated-span pass queued behind this grid launch: it
    // reads nothing this grid writes (with P.gs_merge, nothing before it has
    // seen this grid's completion flag), so its CTAs take the SMs this
    // grid's CTAs leave, and it waits for this grid before it exits.  (Behind the
    // generated-span pass instead, that pass has waited before it let this
    // grid launch; see the end of the kernel.)  No-ops for a plain launch.
    if (!P.prefix_after_gs) {
        asm volatile("griddepcontrol.wait;" ::: "memory");
        // The generated-span pass queued behind this grid claims its items
        // from a counter (sched[2]) and, with merges, reads this grid's
        // completion flag (sched[4]; the last CTA to finish sets it, see the
        // end of the kernel): both are cleared before that pass can launch.
        if (P.gs_after_prefix) {
            if (blockIdx.x == 0 && threadIdx.x == 0) {
                atomicExch(P.sched + 2, 0u);
                if (P.gs_merge) atomicExch(P.sched + 4, 0u);
                __threadfence();
            }
            __syncthreads();
        }
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    }
    const uint32_t tmem = *s_tmem;
    // Item k of the CTA's stream, for a whole warp (item -1 after the last
    // item, -2 when the wait gave up).
    auto take_item = [&](int k) -> ItemInfo {
        const int r = k % kItemRing;
        ItemInfo it;
        if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::IFULL + r), uint32_t(k / kItemRing) & 1u, s_abort, P.err,
                                                   kErrWaitItem))) {
            it.item = -2;
            return it;
        }
        it = s_ring[r];
        __syncwarp();
        if (lane == 0) tc::mbar_arrive(bar(Bb::IEMPTY + r));
        return it;
    };
    // Key block number g of the CTA's stream (counted over all its items)
    // uses S slot g mod NSLOT, for the (g / NSLOT)-th time.
    auto col_s = [](int g) { return uint32_t((g % NSLOT) * C::BN); };
    auto use_of = [](int g) { return uint32_t(g / NSLOT) & 1u; };

    if (warp < 4) {
    // control warpgroup: give registers to the softmax warpgroups
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsControl));
    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        // Two cursors in one thread: K blocks are released by Q K^T and V
        // blocks only later by P V, so each is loaded as soon as its own
        // stage is free instead of in a fixed K, V, K, V order.  The K
        // cursor claims items and posts them; the V cursor takes them from
        // the item ring like the other roles.  Both poll without blocking.
        if (lane == 0) {
            int kpost = 0, vtake = 0;            // items posted / taken by the V cursor
            int kg = 0, vg = 0;                  // K / V blocks issued (CTA-wide)
            int kj = 0, vj = 0;                  // block within the cursor's item
            ItemInfo ki{}, vi{};
            bool k_in = false, v_in = false, k_done = false, v_done = false;
            // The next item is claimed when the K cursor issues the
            // second-to-last block of its item (the claim's latency hides
            // behind the last block's stage wait), so a CTA holds no item it
            // will not start soon: claiming at the item's start left every
            // CTA a whole item ahead, and near the end of the queue some CTAs
            // still held two items while others had none.
            int nxt = int(atomicAdd(P.sched, 1u));
            bool have_nxt = true;
            // a span's tiles read it at about the same time; afterwards its
            // lines go first, keeping the partial states in L2 for the merge
            const uint64_t pol = tc::l2_policy_evict_first();
            uint64_t idle_since = 0;
            uint32_t spins = 0;
            while (!(k_done && v_done)) {
                bool prog = false;
                if (!k_done) {
                    if (!k_in) {
                        const int r = kpost % kItemRing;
                        if (tc::mbar_test_wait(bar(Bb::IEMPTY + r), (uint32_t(kpost / kItemRing) & 1u) ^ 1u)) {
                            if (!have_nxt) nxt = int(atomicAdd(P.sched, 1u));   // an item with no block
                            have_nxt = false;
                            const int item = nxt < tp.n_items ? nxt : -1;
                            ItemInfo inf;
                            inf.item = -1;
                            if (item >= 0) inf = item_info<D>(P, tp, item);
                            s_ring[r] = inf;
                            tc::mbar_arrive(bar(Bb::IFULL + r));
                            ++kpost;
                            prog = true;
                            if (item < 0) {
                                k_done = true;
                            } else {
                                ki = inf;
                                kj = 0;
                                k_in = true;
                            }
                        }
                    }
                    if (k_in && kj == ki.nblk) k_in = false;
                    if (k_in) {
                        const int stg = kg % C::KST;
                        if (tc::mbar_test_wait(bar(Bb::KEMPTY + stg), (uint32_t(kg / C::KST) & 1u) ^ 1u)) {
                            const CUtensorMap* tmk = ki.store == 0 ? &tm_kc : (ki.store == 1 ? &tm_kd : &tm_kx);
                            const int y = int(ki.span_row + ki.k0 + kj * C::BN);
                            tc::mbar_arrive_expect_tx(bar(Bb::KFULL + stg), C::KV_BYTES);
#pragma unroll
                            for (int b = 0; b < C::KB; ++b)
                                tc::tma_load_2d_hint(sbase + C::OFF_K + stg * C::KV_BYTES + b * (C::BN * 128), tmk, b * 64,
                                                     y, bar(Bb::KFULL + stg), pol);
                            ++kg;
                            ++kj;
                            prog = true;
                            if (!have_nxt && kj >= ki.nblk - 1) {
                                nxt = int(atomicAdd(P.sched, 1u));
                                have_nxt = true;
                            }
                        }
                    }
                }
                if (!v_done) {
                    if (!v_in && vtake < kpost) {
                        const int r = vtake % kItemRing;
                        const ItemInfo inf = s_ring[r];
                        tc::mbar_arrive(bar(Bb::IEMPTY + r));
                        ++vtake;
                        prog = true;
                        if (inf.item < 0) {
                            v_done = true;
                        } else {
                            vi = inf;
                            vj = 0;
                            v_in = true;
                        }
                    }
                    if (v_in && vj == vi.nblk) v_in = false;
                    if (v_in && vg < kg) {
                        const int stg = vg % C::VST;
                        if (tc::mbar_test_wait(bar(Bb::VEMPTY + stg), (uint32_t(vg / C::VST) & 1u) ^ 1u)) {
                            const CUtensorMap* tmv = vi.store == 0 ? &tm_vc : (vi.store == 1 ? &tm_vd : &tm_vx);
                            const int y = int(vi.span_row + vi.k0 + vj * C::BN);
                            tc::mbar_arrive_expect_tx(bar(Bb::VFULL + stg), C::KV_BYTES);
#pragma unroll
                            for (int b = 0; b < C::KB; ++b)
                                tc::tma_load_2d_hint(sbase + C::OFF_V + stg * C::KV_BYTES + b * (C::BN * 128), tmv, b * 64,
                                                     y, bar(Bb::VFULL + stg), pol);
                            ++vg;
                            ++vj;
                            prog = true;
                        }
                    }
                }
                // bounded: give up after ~1 s without progress, or when another
                // role did; idle polls back off so they leave the SM's issue
                // slots to the softmax warps
                if (prog) {
                    idle_since = 0;
                    spins = 0;
                } else if (++spins > 4) {
                    __nanosleep(64);
                }
                if (!prog && (spins & 63u) == 0) {
                    if (*s_abort) break;
                    const uint64_t now = tc::globaltimer_ns();
                    if (idle_since == 0) {
                        idle_since = now;
                    } else if (now - idle_since > 1000000000ull) {
                        *s_abort = 1;
                        atomicOr(P.err, kErrWaitProducer);
                        break;
                    }
                }
            }
            // Drain: every issued copy must land before the CTA may exit.
            for (int j = max(0, kg - C::KST); j < kg; ++j) {
                volatile int no_abort = 0;
                tc::mbar_wait(bar(Bb::KFULL + j % C::KST), uint32_t(j / C::KST) & 1u, &no_abort, P.err,
                              kErrWaitDrain);
            }
            for (int j = max(0, vg - C::VST); j < vg; ++j) {
                volatile int no_abort = 0;
                tc::mbar_wait(bar(Bb::VFULL + j % C::VST), uint32_t(j / C::VST) & 1u, &no_abort, P.err,
                              kErrWaitDrain);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ Q K^T issuer
        // The whole warp runs the loop; one elected lane issues the MMAs and
        // their commits.
        const bool leader = tc::elect_one();
        constexpr uint32_t idesc_qk = tc::idesc_bf16_f32(kRows, C::BN, false);
        bool ok = true, committed = false;
        int jg = 0;
        for (int k = 0;; ++k) {
            const ItemInfo it = take_item(k);
            if (it.item < 0) {
                ok = it.item == -1;
                break;
            }
            const int qb = C::NQ == 2 ? (k & 1) : 0;
            const uint32_t quse = uint32_t(C::NQ == 2 ? k >> 1 : k);
            const uint32_t q_addr = sbase + C::OFF_Q + qb * C::Q_BYTES;
            if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::QFULL + qb), quse & 1u, s_abort, P.err, kErrWaitMma))) {
                ok = false;
                break;
            }
            for (int j = 0; j < it.nblk; ++j, ++jg) {
                const int stg = jg % C::KST;
                const int slot = jg % NSLOT;
                // the K block is loaded, and the slot's previous P V is done
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::KFULL + stg), uint32_t(jg / C::KST) & 1u, s_abort,
                                                           P.err, kErrWaitMma)) ||
                    !__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::SFREE + slot), use_of(jg) ^ 1u, s_abort, P.err,
                                                           kErrWaitMma))) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t k_addr = sbase + C::OFF_K + stg * C::KV_BYTES;
                if (leader) {
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk) {
                        const uint64_t a = tc::sw128_desc(q_addr + (kk / 4) * (kRows * 128) + (kk % 4) * 32, 16, 1024);
                        const uint64_t b = tc::sw128_desc(k_addr + (kk / 4) * (C::BN * 128) + (kk % 4) * 32, 16, 1024);
                        tc::mma_f16_ss(tmem + col_s(jg), a, b, idesc_qk, kk > 0 ? 1u : 0u);
                    }
                    tc::mma_commit(bar(Bb::SFULL + slot));
                    tc::mma_commit(bar(Bb::KEMPTY + stg));
                    if (j == it.nblk - 1) tc::mma_commit(bar(Bb::QEMPTY + qb));
                }
                committed = true;
            }
            if (!ok) break;
            if (it.nblk == 0 && leader) tc::mma_commit(bar(Bb::QEMPTY + qb));
        }
        if (!ok && committed && leader) {
            // Let the MMAs already issued finish before TMEM is freed.
            tc::mma_commit(bar(Bb::DRAIN));
            volatile int no_abort = 0;
            tc::mbar_wait(bar(Bb::DRAIN), 0, &no_abort, P.err, kErrWaitDrain);
        }
    } else if (warp == kPvWarp) {
        // ------------------------------------------------ P V issuer
        const bool leader = tc::elect_one();
        constexpr uint32_t idesc_pv = tc::idesc_bf16_f32(kRows, D, true);
        bool ok = true, committed = false;
        int jg = 0;
        for (int k = 0;; ++k) {
            const ItemInfo it = take_item(k);
            if (it.item < 0) {
                ok = it.item == -1;
                break;
            }
            // The softmax has read the previous item's O.  Waited for at every
            // item, an empty one included, so that ODONE never completes a
            // second phase before the softmax has seen the first (a parity
            // wait cannot tell them apart).
            if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::OFREE), (uint32_t(k) & 1u) ^ 1u, s_abort, P.err,
                                                       kErrWaitMma))) {
                ok = false;
                break;
            }
            for (int j = 0; j < it.nblk; ++j, ++jg) {
                const int stg = jg % C::VST;
                const int slot = jg % NSLOT;
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::PFULL + slot), use_of(jg), s_abort, P.err,
                                                           kErrWaitMma)) ||
                    !__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::VFULL + stg), uint32_t(jg / C::VST) & 1u, s_abort,
                                                           P.err, kErrWaitMma))) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t v_addr = sbase + C::OFF_V + stg * C::KV_BYTES;
                const uint32_t p_col = tmem + col_s(jg);
                if (leader) {
#pragma unroll
                    for (int kk = 0; kk < C::BN / 16; ++kk) {
                        // 16 keys of P: two bf16 per TMEM column; the first
                        // half's P sits at the start of the slot, the second
                        // half's at its middle
                        const uint32_t a = p_col + (kk / (C::KPT / 16)) * C::KPT + (kk % (C::KPT / 16)) * 8;
                        const uint64_t b = tc::sw128_desc(v_addr + kk * 16 * 128, C::BN * 128, 1024);
                        mma_f16_ts(tmem + C::COL_O, a, b, idesc_pv, (j > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(bar(Bb::SFREE + slot));
                    tc::mma_commit(bar(Bb::VEMPTY + stg));
                }
                committed = true;
            }
            if (!ok) break;
            if (leader) tc::mma_commit(bar(Bb::ODONE));
        }
        if (!ok && committed && leader) {
            tc::mma_commit(bar(Bb::DRAIN + 1));
            volatile int no_abort = 0;
            tc::mbar_wait(bar(Bb::DRAIN + 1), 0, &no_abort, P.err, kErrWaitDrain);
        }
    } else if (warp == 2) {
        // ------------------------------------------------ Q gather
        // Rows no item fills keep finite values: zero every buffer once.
        for (uint32_t off = uint32_t(lane) * 16; off < C::NQ * C::Q_BYTES; off += 32 * 16)
            *reinterpret_cast<uint4*>(smem + C::OFF_Q + off) = make_uint4(0, 0, 0, 0);
        __syncwarp();
        for (int k = 0;; ++k) {
            const ItemInfo it = take_item(k);
            if (it.item < 0) break;
            const int nrows = it.nblk > 0 ? it.nseq * P.G : 0;   // an empty split reads no Q
            const int qb = C::NQ == 2 ? (k & 1) : 0;
            const uint32_t quse = uint32_t(C::NQ == 2 ? k >> 1 : k);
            if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::QEMPTY + qb), (quse & 1u) ^ 1u, s_abort, P.err, kErrWaitQ)))
                break;
            const uint32_t q_s = sbase + C::OFF_Q + qb * C::Q_BYTES;
#pragma unroll 1
            for (int row = lane; row < nrows; row += 32) {
                const int s = P.group_seqs[it.first + row / P.G];
                const int hq = it.h * P.G + row % P.G;
                const uint16_t* src = P.q + (long(s) * P.Hq + hq) * D;
                const uint32_t dst = q_s + row * 128;
#pragma unroll
                for (int c = 0; c < D / 8; ++c)
                    tc::cp_async16(dst + (c / 8) * (kRows * 128) + (((c % 8) ^ (row % 8)) * 16), src + c * 8);
            }
            tc::cp_async_wait_all();
            tc::fence_proxy_async_smem();
            tc::mbar_arrive(bar(Bb::QFULL + qb));
        }
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsSoftmax));
        // ------------------------------------------------ softmax / epilogue
        const int wg = (warp - 4) / 4;                 // 0: first half of each block's keys, 1: second half
        const int quarter = warp & 3;                  // TMEM lane quarter this warp may access
        const uint32_t lane_base = uint32_t(quarter * 32) << 16;
        float* xmax = reinterpret_cast<float*>(smem + C::OFF_X);          // [2][2][128]
        float* xl = xmax + 2 * 2 * kRows;                                 // [2][2][128]
        const float c = P.scale_log2;
        const float2 c2 = make_float2(c, c);
        const float neg = c >= 0.f ? -INFINITY : INFINITY;     // a raw logit that weighs nothing
        const bool zero_scale = c == 0.f;                      // then neg * c is not -inf
        constexpr int KPT = C::KPT;                    // keys of this thread per block
        constexpr int SEG = KPT / 2;                   // keys per row-sum segment
        const int row = quarter * 32 + lane;           // == TMEM lane of this thread's row
        int jg = 0;
        // An item's epilogue (its partial states out of O, then O freed).
        // For d = 256 (64-key blocks, half as long) it is deferred past the
        // next item's first block, whose softmax then runs while the item's
        // last P V completes (a Gemma-3-4B-shaped sweep +1.4%); for d <= 128
        // that held O, and so the next item's first P V, too long for the
        // three S slots to cover (the ladder -1.3%).  The item's state:
        constexpr bool kDefer = D == 256;
        bool pend = false, pend_full = false, pend_rows = false;
        int pend_k = 0, pend_idx = -1;                 // pend_idx: -1 for a row outside the tile
        float pend_m = 0.f, pend_l = 0.f;
        auto epilogue = [&]() -> bool {
            pend = false;
            // Every thread waits for the item's O before it frees it, so
            // arrivals of one item never land in an earlier item's phase.
            if (!__all_sync(0xffffffffu,
                            tc::mbar_wait(bar(Bb::ODONE), uint32_t(pend_k) & 1u, s_abort, P.err, kErrWaitSoftmax)))
                return false;
            tc::tc_fence_after();
            float* xb = xl + (pend_k & 1) * (2 * kRows);
            if (pend_full) {
                if (pend_rows) {
                    // Each thread holds its row's half of O.  Stores of one
                    // value per thread would touch 32 rows (lines) per
                    // instruction, so the warp stages 16 columns of its 32
                    // rows at a time in shared memory and stores them as 8
                    // rows x 64 contiguous bytes per instruction (16-byte
                    // units rotated by row pair, so neither side conflicts).
                    int ridx[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) ridx[i] = __shfl_sync(0xffffffffu, pend_idx, i * 8 + lane / 4);
                    float* stg = reinterpret_cast<float*>(smem + C::OFF_STG + (warp - 4) * C::STG_BYTES);
                    const int u = lane & 3;
#pragma unroll
                    for (int q = 0; q < C::OCH / 32; ++q) {
                        float v[32];
                        tc::tmem_ld32(tmem + lane_base + C::COL_O + wg * C::OCH + q * 32, v);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
#pragma unroll
                            for (int w = 0; w < 4; ++w) {
                                const int slot = (w + (lane >> 1)) & 3;
                                *reinterpret_cast<float4*>(stg + lane * 16 + slot * 4) =
                                    make_float4(v[h * 16 + w * 4], v[h * 16 + w * 4 + 1], v[h * 16 + w * 4 + 2],
                                                v[h * 16 + w * 4 + 3]);
                            }
                            __syncwarp();
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const int r = i * 8 + lane / 4;
                                const float4 x =
                                    *reinterpret_cast<const float4*>(stg + r * 16 + ((u + (r >> 1)) & 3) * 4);
                                if (ridx[i] >= 0)
                                    *reinterpret_cast<float4*>(P.ws_o + size_t(ridx[i]) * D + wg * C::OCH + q * 32 +
                                                               h * 16 + u * 4) = x;
                            }
                            __syncwarp();
                        }
                    }
                }
                xb[wg * kRows + row] = pend_l;
                tc::mbar_arrive(bar(Bb::LXCH));
                if (!__all_sync(0xffffffffu,
                                tc::mbar_wait(bar(Bb::LXCH), uint32_t(pend_k) & 1u, s_abort, P.err, kErrWaitSoftmax)))
                    return false;
                if (wg == 0 && pend_idx >= 0) P.ws_ml[pend_idx] = make_float2(pend_m, xb[row] + xb[kRows + row]);
            } else {
                // an empty split: a state with no keys (still one exchange
                // round, so every item moves the exchange barrier once)
                tc::mbar_arrive(bar(Bb::LXCH));
                if (!__all_sync(0xffffffffu,
                                tc::mbar_wait(bar(Bb::LXCH), uint32_t(pend_k) & 1u, s_abort, P.err, kErrWaitSoftmax)))
                    return false;
                if (wg == 0 && pend_idx >= 0) P.ws_ml[pend_idx] = make_float2(-INFINITY, 0.f);
            }
            tc::tc_fence_before();
            tc::mbar_arrive(bar(Bb::OFREE));
            return true;
        };
        bool ok = true;
        for (int k = 0;; ++k) {
            const ItemInfo it = take_item(k);
            if (it.item < 0) {
                ok = it.item == -1;
                break;
            }
            const int nrows = it.nseq * P.G;
            const bool rows = quarter * 32 < nrows;    // warp-uniform
            const bool valid = row < nrows;
            // the row's sequence: loaded now, needed only at the item's end
            const int seq = valid ? P.group_seqs[it.first + row / P.G] : 0;
            // delta mode: the bits of the positions this row's donor
            // encodes (they come from the delta rows, not from this span)
            const uint32_t* mrow = nullptr;
            if (it.masked && valid) {
                const int mid = P.group_mask[it.first + row / P.G];
                if (mid > 0)
                    mrow = P.dmask + size_t(((long(it.prompt) * P.Dst + (mid - 1)) * P.N + P.layer) * P.Hkv + it.h) *
                                         size_t(P.delta_w32);
            }
            // row sum kept per segment of this thread's keys (two), added at
            // the item's end
            float m_run = -INFINITY, l_seg0 = 0.f, l_seg1 = 0.f;
            for (int j = 0; j < it.nblk; ++j, ++jg) {
                const int slot = jg % NSLOT;
                // waits are made warp-uniform: tcgen05.ld/st are warp-collective
                if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::SFULL + slot), use_of(jg), s_abort, P.err,
                                                           kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                const uint32_t s_col = tmem + lane_base + col_s(jg) + wg * KPT;
                const int kbase = it.k0 + j * C::BN + wg * KPT;
                float s[KPT];
                float e0 = 0.f;
                // keys of this half that do not count: past the split's end,
                // and the positions this row's donor encodes
                uint32_t dead[KPT / 32];
                bool any_dead = false;
                if (rows) {
                    tc::tc_fence_after();
#pragma unroll
                    for (int q = 0; q < KPT / 32; ++q) {
                        float v[32];
                        tc::tmem_ld32(s_col + q * 32, v);
#pragma unroll
                        for (int i = 0; i < 32; ++i) s[q * 32 + i] = v[i];
                    }
                    uint32_t anyd = 0u;
#pragma unroll
                    for (int q = 0; q < KPT / 32; ++q) {
                        const int live = it.k1 - (kbase + 32 * q);
                        dead[q] = live >= 32 ? 0u : (live <= 0 ? 0xffffffffu : (0xffffffffu << live));
                        if (mrow) dead[q] |= __ldg(mrow + (kbase >> 5) + q);
                        anyd |= dead[q];
                    }
                    any_dead = __any_sync(0xffffffffu, anyd != 0u);
                    tc::tmem_wait_ld();
                    if (any_dead) {
#pragma unroll
                        for (int i = 0; i < KPT; ++i)
                            if ((dead[i >> 5] >> (i & 31)) & 1u) s[i] = neg;
                    }
                    // extreme of this half's raw logits (max for c >= 0)
                    float e1 = s[1], e2 = s[2], e3 = s[3];
                    e0 = s[0];
                    if (c >= 0.f) {
#pragma unroll
                        for (int i = 4; i < KPT; i += 4) {
                            e0 = fmaxf(e0, s[i]);
                            e1 = fmaxf(e1, s[i + 1]);
                            e2 = fmaxf(e2, s[i + 2]);
                            e3 = fmaxf(e3, s[i + 3]);
                        }
                        e0 = fmaxf(fmaxf(e0, e1), fmaxf(e2, e3));
                    } else {
#pragma unroll
                        for (int i = 4; i < KPT; i += 4) {
                            e0 = fminf(e0, s[i]);
                            e1 = fminf(e1, s[i + 1]);
                            e2 = fminf(e2, s[i + 2]);
                            e3 = fminf(e3, s[i + 3]);
                        }
                        e0 = fminf(fminf(e0, e1), fminf(e2, e3));
                    }
                }
                // the two halves of the block trade their extremes (only the
                // two warps holding this lane quarter's rows meet here)
                float* xm = xmax + (jg & 1) * (2 * kRows);
                xm[wg * kRows + row] = e0;
                const uint32_t xch = bar(Bb::XCH + 4 * (jg & 1) + quarter);
                tc::mbar_arrive(xch);
                if (!__all_sync(0xffffffffu,
                                tc::mbar_wait(xch, uint32_t(jg >> 1) & 1u, s_abort, P.err, kErrWaitSoftmax))) {
                    ok = false;
                    break;
                }
                if (rows) {
                    const float eo = xm[(wg ^ 1) * kRows + row];
                    const float mc = (c >= 0.f ? fmaxf(e0, eo) : fminf(e0, eo)) * c;   // block max, log2 units
                    float alpha = 1.f;
                    bool resc = false;
                    if (mc > m_run + kTau) {
                        alpha = ex2(m_run - mc);
                        resc = j > 0;
                        m_run = mc;
                    }
                    // no live key yet (every earlier key of the row dead): any
                    // finite reference makes the dead keys' weights 0
                    const float mref = m_run == -INFINITY ? 0.f : m_run;
                    const float2 nm2 = make_float2(-mref, -mref);
                    // per segment: exponentials, the segment's row sum, and
                    // its P (bf16 pairs) stored over the first columns of
                    // this half of the slot
#pragma unroll
                    for (int g = 0; g < 2; ++g) {
                        float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
                        uint32_t pk[SEG / 2];
#pragma unroll
                        for (int i = 0; i < SEG / 2; ++i) {
                            const int pi = g * (SEG / 2) + i;
                            const float2 z = __ffma2_rn(make_float2(s[2 * pi], s[2 * pi + 1]), c2, nm2);
                            float2 e = make_float2(ex2(z.x), ex2(z.y));
                            if (any_dead && zero_scale) {
                                e.x = ((dead[(2 * pi) >> 5] >> ((2 * pi) & 31)) & 1u) ? 0.f : e.x;
                                e.y = ((dead[(2 * pi + 1) >> 5] >> ((2 * pi + 1) & 31)) & 1u) ? 0.f : e.y;
                            }
                            if (i & 1)
                                acc1 = __fadd2_rn(acc1, e);
                            else
                                acc0 = __fadd2_rn(acc0, e);
                            const __nv_bfloat162 h2 = __floats2bfloat162_rn(e.x, e.y);
                            pk[i] = *reinterpret_cast<const uint32_t*>(&h2);
                        }
                        const float ls = (acc0.x + acc1.x) + (acc0.y + acc1.y);
                        if (g == 0)
                            l_seg0 = l_seg0 * alpha + ls;
                        else
                            l_seg1 = l_seg1 * alpha + ls;
                        store_p(s_col + g * (SEG / 2), pk);
                    }
                    if (__any_sync(0xffffffffu, resc)) {
                        // O must hold P V of every earlier block of this item
                        const int jp = jg - 1;
                        if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(Bb::SFREE + jp % NSLOT), use_of(jp), s_abort,
                                                                   P.err, kErrWaitSoftmax))) {
                            ok = false;
                            break;
                        }
                        tc::tc_fence_after();
                        const float2 a2 = make_float2(resc ? alpha : 1.f, resc ? alpha : 1.f);
#pragma unroll
                        for (int q = 0; q < C::OCH / 32; ++q) {
                            float v[32];
                            const uint32_t ta = tmem + lane_base + C::COL_O + wg * C::OCH + q * 32;
                            tc::tmem_ld32(ta, v);
                            tc::tmem_wait_ld();
#pragma unroll
                            for (int i = 0; i < 32; i += 2) {
                                const float2 r = __fmul2_rn(make_float2(v[i], v[i + 1]), a2);
                                v[i] = r.x;
                                v[i + 1] = r.y;
                            }
                            tc::tmem_st32(ta, v);
                        }
                    }
                    tc::tmem_wait_st();
                }
                tc::tc_fence_before();
                tc::mbar_arrive(bar(Bb::PFULL + slot));
                // the previous item's epilogue, now that this item's first P
                // is out
                if (kDefer && pend && !epilogue()) {
                    ok = false;
                    break;
                }
            }
            if (!ok) break;
            // an item with no block has nothing to overlap with
            if (pend && !epilogue()) {
                ok = false;
                break;
            }
            // ---- this item's partial state: written after the next item's
            // first block ----
            const int orow = seq * P.Hq + it.h * P.G + row % P.G;
            // (a partial-state index fits in 32 bits: the workspace holds 16 x
            // rows x 520 bytes, far below 2^31 rows of device memory)
            pend_idx = valid ? int(size_t(it.split) * P.B * P.Hq + size_t(orow)) : -1;
            pend_full = it.nblk > 0;
            pend_rows = rows;
            pend_k = k;
            // a row's sum: its segments' sums in key order, then (in the
            // epilogue) the two halves
            pend_m = m_run;
            pend_l = l_seg0 + l_seg1;
            pend = true;
            if (!kDefer && !epilogue()) {
                ok = false;
                break;
            }
        }
        if (ok && pend) epilogue();
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    if (warp == 1) tc::tmem_dealloc(tmem, kTmemCols);
    if (P.prefix_after_gs) {
        // This CTA's work is done: the merge queued behind this grid may
        // launch (it waits for the whole grid before it reads anything).
        // Every CTA of this grid is running by the time all of them have
        // signalled, so the merge's CTAs never hold an SM it still needs.
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        // Launched right behind the generated-span pass, this grid may start
        // while that pass's last CTAs still run (it reads nothing they
        // write); waiting for it here makes this grid's completion imply that
        // pass's, so the merge that follows sees both.
        asm volatile("griddepcontrol.wait;" ::: "memory");
    }
    // The last CTA to finish resets the work counter for the next launch
    // (every CTA's claims have returned before it gets here, so they are
    // performed).  With merges in the generated-span pass it then sets the
    // completion flag: every CTA fenced its partial states (written before
    // the barrier above) before it counted itself, so a reader that sees
    // the flag and then fences sees them all.
    if (threadIdx.x == 0) {
        if (P.gs_merge) __threadfence();
        if (atomicAdd(P.sched + 1, 1u) == gridDim.x - 1) {
            atomicExch(P.sched, 0u);
            atomicExch(P.sched + 1, 0u);
            if (P.gs_merge) {
                __threadfence();
                atomicExch(P.sched + 4, 1u);
            }
        }
    }
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

template <int D, bool SHORT>
int launch_d(const TcParams& tp, const CUtensorMap* m, cudaStream_t st, bool overlap_previous) {
    using C = Cfg<D, SHORT>;
    static int sms = 0;
    if (!sms) {
        cudaFuncSetAttribute(prefix_tc_kernel<D, SHORT>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    const unsigned grid = unsigned(tp.n_items < sms ? tp.n_items : sms);
    if (!overlap_previous) {
        prefix_tc_kernel<D, SHORT><<<grid, kThreads, C::SMEM, st>>>(m[0], m[1], m[2], m[3], m[4], m[5], tp);
        return 0;
    }
    // programmatic dependent launch: CTAs may start as the previous grid's
    // CTAs retire
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::SMEM;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return int(cudaLaunchKernelEx(&cfg, prefix_tc_kernel<D, SHORT>, m[0], m[1], m[2], m[3], m[4], m[5], tp));
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

int prefix_tc_box_rows(int d) {
    return d == 64 ? Cfg<64>::BN : (d == 128 ? Cfg<128>::BN : Cfg<256>::BN);
}

int prefix_tc_splits(int d, int p_vis, int max_splits, int* bounds) {
    // Splits depend only on the visible span length (and the cap), so a
    // row's arithmetic never depends on which other rows share its tile or
    // launch.  Every item gathers its tile's queries and stores its partial
    // states, so long items move fewer bytes; but a launch ends as unevenly
    // as its last items are long.  So a span's first split is
    // kPrefixFirstSplitKeys keys and the rest kPrefixSplitKeys: the
    // split-major item order hands out every span's long first split before
    // the short ones, and the launch ends on short items.  Past the cap, the
    // blocks are shared out evenly.
    const int bn = prefix_tc_box_rows(d);
    const int nb = (p_vis + bn - 1) / bn;
    const int first = kPrefixFirstSplitKeys / bn, rest = kPrefixSplitKeys / bn;
    const int ns_full = nb <= first ? 1 : 1 + (nb - first + rest - 1) / rest;
    bounds[0] = 0;
    if (ns_full <= max_splits) {
        for (int i = 0; i < ns_full; ++i) {
            const int b = bounds[i] + (i == 0 ? first : rest) * bn;
            bounds[i + 1] = b < p_vis ? b : p_vis;
        }
        return ns_full;
    }
    const int ns = max_splits;
    for (int i = 0; i < ns; ++i) {
        const int blocks = nb / ns + (i < nb % ns ? 1 : 0);
        const int b = bounds[i] + blocks * bn;
        bounds[i + 1] = b < p_vis ? b : p_vis;
    }
    return ns;
}

int launch_prefix_tc(const AttnParams& p, const void* maps, const int* bounds, int delta_keys, void* stream,
                     bool overlap_previous) {
    const CUtensorMap* m = static_cast<const CUtensorMap*>(maps);
    const int n_span_items = p.n_span_tiles * p.Hkv * p.nsp;
    TcParams tp{};
    tp.a = p;
    for (int i = 0; i <= p.nsp && i <= kMaxPrefixSplits; ++i) tp.sb[i] = bounds[i];
    tp.delta_keys = delta_keys;
    tp.n_span_items = n_span_items;
    tp.n_items = n_span_items + (p.n_tiles - p.n_span_tiles) * p.Hkv * p.nsd;
    if (tp.n_items <= 0) return 0;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int r = int(cudaErrorInvalidValue);
    // every item of at most four key blocks: the short-item ring layout
    const int bn = prefix_tc_box_rows(p.D);
    const bool short_items = p.D <= 128 && bounds[1] <= 4 * bn && (p.nsd == 0 || delta_keys <= 4 * bn);
    switch (p.D) {
        case 64:
            r = short_items ? launch_d<64, true>(tp, m, st, overlap_previous)
                            : launch_d<64, false>(tp, m, st, overlap_previous);
            break;
        case 128:
            r = short_items ? launch_d<128, true>(tp, m, st, overlap_previous)
                            : launch_d<128, false>(tp, m, st, overlap_previous);
            break;
        case 256: r = launch_d<256, false>(tp, m, st, overlap_previous); break;
        default: break;
    }
    if (r != 0) return r;
    return int(cudaGetLastError());
}

}  // namespace splice
