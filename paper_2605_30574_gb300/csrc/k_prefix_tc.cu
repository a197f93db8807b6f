// Tensor-core prompt-span pass (tcgen05 + TMEM, TMA-fed).
//
// Every sequence that reads the same (prompt, source) span at a (layer,
// step) -- a group of the descriptor's table -- shares that span's K/V.  For
// one kv head h, the G query rows of every sequence of the group are stacked
// into 128-row tiles, so Q K^T and P V over the span are real dense
// contractions: M = 128 stacked rows, N = a block of keys (or d), K = d (or
// keys).  One CTA handles one (row tile, kv head, key split):
//
//   warp 0        TMA producer: K and V key blocks of the span -> smem ring
//   warp 1        MMA issuer (one lane): S = Q K^T into TMEM (two buffers),
//                 O += P V into TMEM; owns the TMEM allocation
//   warps 2..5    softmax / epilogue, one row per thread: S from TMEM, online
//                 softmax with a lazily moved reference max, P (bf16) to smem,
//                 O rescale in TMEM when the reference moves; at the end the
//                 partial state (m, l, o) of each row goes to the workspace
//
// The merge kernel combines these partials with those of the generated span
// (and the ZERO closed form), exactly like the CUDA-core partials.
//
// Every wait is bounded: a wait that runs out sets a CTA abort flag and an
// error bit in the descriptor's error word; all roles then leave their loops,
// outstanding TMA copies and MMAs are waited for (bounded), TMEM is freed and
// the CTA exits without writing results.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>

#include "splice_internal.h"
#include "tc_ptx.cuh"

namespace splice {
namespace {

constexpr int kRows = 128;          // MMA M
constexpr int kThreads = 192;       // 6 warps
constexpr uint32_t kTmemCols = 512;
constexpr float kTau = 8.0f;        // lazy rescale threshold, log2 units

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Error codes recorded in the descriptor's error word.
constexpr unsigned kErrWaitProducer = 0x1, kErrWaitMma = 0x2, kErrWaitSoftmax = 0x4, kErrWaitDrain = 0x8;

template <int D>
struct Cfg {
    static constexpr int BN = D == 256 ? 64 : 128;          // keys per block
    static constexpr int STAGES = D == 64 ? 3 : 2;
    static constexpr int KB = D / 64;                         // 64-wide K blocks of Q / K tile
    static constexpr uint32_t Q_BYTES = kRows * D * 2;
    static constexpr uint32_t KV_BYTES = BN * D * 2;          // one K (or V) block
    static constexpr uint32_t P_BYTES = kRows * BN * 2;
    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_K = OFF_Q + Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr uint32_t OFF_P = OFF_V + STAGES * KV_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_P + P_BYTES;
    static constexpr uint32_t SMEM = OFF_BAR + 256 + 1024;    // + barriers, + alignment slack
    // TMEM columns: S buffers at 0 and BN, O at 2 BN.
    static constexpr uint32_t COL_S0 = 0, COL_S1 = BN, COL_O = 2 * BN;
    static_assert(2 * BN + D <= int(kTmemCols), "TMEM budget");
    static_assert(SMEM <= 227 * 1024, "shared memory budget");
};

struct TcParams {
    AttnParams a;
    int nsplit;
    int split_keys;     // keys per split (multiple of BN)
};

// Barrier slots (8 bytes each) in the barrier area.
enum : int {
    B_KFULL = 0,    // [STAGES]
    B_KEMPTY = 4,   // [STAGES]
    B_VFULL = 8,    // [STAGES]
    B_VEMPTY = 12,  // [STAGES]
    B_SFULL = 16,   // [2]
    B_SFREE = 18,   // [2]
    B_PFULL = 20,
    B_PEMPTY = 21,
    B_ODONE = 22,
    B_QREADY = 23,
    B_COUNT = 24
};

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

    // ---- work item: (tile, kv head, split) ----
    const int tile = blockIdx.x % P.n_tiles;
    const int hs = blockIdx.x / P.n_tiles;
    const int split = hs % tp.nsplit;
    const int h = hs / tp.nsplit;
    const int4 tl = reinterpret_cast<const int4*>(P.tiles)[tile];
    const int grp = tl.x, first = tl.y, nseq = tl.z;
    const int nrows = nseq * P.G;
    const int prompt = P.group_prompt[grp];
    const int code = P.group_src[grp];
    const bool donor = code != int(SPLICE_SRC_CLEAN);
    long span;
    if (!donor) {
        span = (long(prompt) * P.N + P.layer) * P.Hkv + h;
    } else {
        const int st = P.slot_stored[code - int(SPLICE_SRC_DONOR0)];
        span = ((long(prompt) * P.Dst + st) * P.N + P.layer) * P.Hkv + h;
    }
    const int row0 = int(span * P.Tp);           // first row of the span in the store's 2D view
    const int k0 = P.p_lo + split * tp.split_keys;
    const int k1 = min(P.p_hi, k0 + tp.split_keys);
    const int nblk = k1 > k0 ? (k1 - k0 + C::BN - 1) / C::BN : 0;
    const CUtensorMap* tmk = donor ? &tm_kd : &tm_kc;
    const CUtensorMap* tmv = donor ? &tm_vd : &tm_vc;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::STAGES; ++i) {
            tc::mbar_init(bar(B_KFULL + i), 1);
            tc::mbar_init(bar(B_KEMPTY + i), 1);
            tc::mbar_init(bar(B_VFULL + i), 1);
            tc::mbar_init(bar(B_VEMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            tc::mbar_init(bar(B_SFULL + i), 1);
            tc::mbar_init(bar(B_SFREE + i), kRows);
        }
        tc::mbar_init(bar(B_PFULL), kRows);
        tc::mbar_init(bar(B_PEMPTY), 1);
        tc::mbar_init(bar(B_ODONE), 1);
        tc::mbar_init(bar(B_QREADY), kRows);
        *s_abort = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(tmk);
        tc::prefetch_tmap(tmv);
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
            int issued_k = 0, issued_v = 0;
            for (int j = 0; j < nblk && !*s_abort; ++j) {
                const int stg = j % C::STAGES;
                const uint32_t use = uint32_t(j / C::STAGES);
                const int y = row0 + k0 + j * C::BN;
                if (!tc::mbar_wait(bar(B_KEMPTY + stg), (use & 1u) ^ 1u, s_abort, P.err, kErrWaitProducer)) break;
                tc::mbar_arrive_expect_tx(bar(B_KFULL + stg), C::KV_BYTES);
#pragma unroll
                for (int b = 0; b < C::KB; ++b)
                    tc::tma_load_2d(sbase + C::OFF_K + stg * C::KV_BYTES + b * (C::BN * 128), tmk, b * 64, y,
                                    bar(B_KFULL + stg));
                issued_k = j + 1;
                if (!tc::mbar_wait(bar(B_VEMPTY + stg), (use & 1u) ^ 1u, s_abort, P.err, kErrWaitProducer)) break;
                tc::mbar_arrive_expect_tx(bar(B_VFULL + stg), C::KV_BYTES);
#pragma unroll
                for (int b = 0; b < C::KB; ++b)
                    tc::tma_load_2d(sbase + C::OFF_V + stg * C::KV_BYTES + b * (C::BN * 128), tmv, b * 64, y,
                                    bar(B_VFULL + stg));
                issued_v = j + 1;
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
            const uint32_t q_addr = sbase + C::OFF_Q, p_addr = sbase + C::OFF_P;
            bool ok = tc::mbar_wait(bar(B_QREADY), 0, s_abort, P.err, kErrWaitMma);
            bool committed = false;
            auto pv = [&](int j) -> bool {
                const int stg = j % C::STAGES;
                if (!tc::mbar_wait(bar(B_PFULL), uint32_t(j) & 1u, s_abort, P.err, kErrWaitMma)) return false;
                if (!tc::mbar_wait(bar(B_VFULL + stg), uint32_t(j / C::STAGES) & 1u, s_abort, P.err, kErrWaitMma))
                    return false;
                tc::tc_fence_after();
                const uint32_t v_addr = sbase + C::OFF_V + stg * C::KV_BYTES;
#pragma unroll
                for (int kk = 0; kk < C::BN / 16; ++kk) {
                    // A = P rows x 16 keys (K-major, 64-key blocks of 128 x 128 B);
                    // B = V 16 keys x d (MN-major: 64-wide d blocks BN x 128 B apart).
                    const uint64_t a = tc::sw128_desc(p_addr + (kk / 4) * (kRows * 128) + (kk % 4) * 32, 16, 1024);
                    const uint64_t b = tc::sw128_desc(v_addr + kk * 16 * 128, C::BN * 128, 1024);
                    tc::mma_f16_ss(tmem + C::COL_O, a, b, idesc_pv, (j > 0 || kk > 0) ? 1u : 0u);
                }
                tc::mma_commit(bar(B_PEMPTY));
                tc::mma_commit(bar(B_VEMPTY + stg));
                committed = true;
                return true;
            };
            for (int j = 0; ok && j < nblk; ++j) {
                const int stg = j % C::STAGES;
                const int sb = j & 1;
                if (!tc::mbar_wait(bar(B_KFULL + stg), uint32_t(j / C::STAGES) & 1u, s_abort, P.err, kErrWaitMma) ||
                    !tc::mbar_wait(bar(B_SFREE + sb), (uint32_t(j / 2) & 1u) ^ 1u, s_abort, P.err, kErrWaitMma)) {
                    ok = false;
                    break;
                }
                tc::tc_fence_after();
                const uint32_t k_addr = sbase + C::OFF_K + stg * C::KV_BYTES;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint64_t a = tc::sw128_desc(q_addr + (kk / 4) * (kRows * 128) + (kk % 4) * 32, 16, 1024);
                    const uint64_t b = tc::sw128_desc(k_addr + (kk / 4) * (C::BN * 128) + (kk % 4) * 32, 16, 1024);
                    tc::mma_f16_ss(tmem + (sb ? C::COL_S1 : C::COL_S0), a, b, idesc_qk, kk > 0 ? 1u : 0u);
                }
                tc::mma_commit(bar(B_SFULL + sb));
                tc::mma_commit(bar(B_KEMPTY + stg));
                committed = true;
                if (j >= 1 && !pv(j - 1)) {
                    ok = false;
                    break;
                }
            }
            if (ok && nblk > 0) ok = pv(nblk - 1);
            tc::mma_commit(bar(B_ODONE));
            if (!ok && committed) {
                // Let the MMAs already issued finish before TMEM is freed.
                volatile int no_abort = 0;
                tc::mbar_wait(bar(B_ODONE), 0, &no_abort, P.err, kErrWaitDrain);
            }
        }
    } else {
        // ------------------------------------------------ softmax / epilogue
        const int r = threadIdx.x - 64;                // 0..127: row of the tile
        const int quarter = warp & 3;                  // TMEM lane quarter this warp may access
        const int row = quarter * 32 + lane;           // == TMEM lane of this thread's row
        const bool valid = row < nrows;
        (void)r;
        // Q row -> smem (K-major, 128-byte swizzle), zero for padding rows.
        long out_row = 0;
        {
            uint8_t* q_s = smem + C::OFF_Q;
            if (valid) {
                const int s = P.group_seqs[first + row / P.G];
                const int hq = h * P.G + row % P.G;
                out_row = long(s) * P.Hq + hq;
                const uint4* src = reinterpret_cast<const uint4*>(P.q + out_row * D);
#pragma unroll
                for (int c = 0; c < D / 8; ++c) {
                    const uint4 v = src[c];
                    *reinterpret_cast<uint4*>(q_s + (c / 8) * (kRows * 128) + row * 128 + (((c % 8) ^ (row % 8)) * 16)) = v;
                }
            } else {
#pragma unroll
                for (int c = 0; c < D / 8; ++c)
                    *reinterpret_cast<uint4*>(q_s + (c / 8) * (kRows * 128) + row * 128 + (((c % 8) ^ (row % 8)) * 16)) =
                        make_uint4(0, 0, 0, 0);
            }
            tc::fence_proxy_async_smem();
            tc::mbar_arrive(bar(B_QREADY));
        }
        const float c = P.scale_log2;
        float m_run = -INFINITY, l_run = 0.f;
        const uint32_t lane_base = uint32_t(quarter * 32) << 16;
        uint8_t* p_s = smem + C::OFF_P;
        bool ok = true;
        for (int j = 0; j < nblk; ++j) {
            const int sb = j & 1;
            // waits are made warp-uniform: the tcgen05.ld/st below are warp-collective
            if (!__all_sync(0xffffffffu,
                            tc::mbar_wait(bar(B_SFULL + sb), uint32_t(j / 2) & 1u, s_abort, P.err, kErrWaitSoftmax))) {
                ok = false;
                break;
            }
            tc::tc_fence_after();
            float s[C::BN];
#pragma unroll
            for (int q = 0; q < C::BN / 32; ++q) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + (sb ? C::COL_S1 : C::COL_S0) + q * 32, v);
#pragma unroll
                for (int i = 0; i < 32; ++i) s[q * 32 + i] = v[i];
            }
            tc::tmem_wait_ld();
            tc::tc_fence_before();
            tc::mbar_arrive(bar(B_SFREE + sb));
            // mask keys past the split end, then the block's reference max
            const int kbase = k0 + j * C::BN;
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < C::BN; ++i) {
                float z = s[i] * c;
                z = (kbase + i < k1) ? z : -INFINITY;
                s[i] = z;
                mx = fmaxf(mx, z);
            }
            float alpha = 1.f;
            bool rescale = false;
            if (mx > m_run + kTau) {
                alpha = ex2(m_run - mx);
                rescale = j > 0;
                m_run = mx;
            }
            float lsum = 0.f;
            uint32_t pk[C::BN / 2];
#pragma unroll
            for (int i = 0; i < C::BN / 2; ++i) {
                const float a = ex2(s[2 * i] - m_run);
                const float b = ex2(s[2 * i + 1] - m_run);
                lsum += a + b;
                const __nv_bfloat162 h2 = __floats2bfloat162_rn(a, b);
                pk[i] = *reinterpret_cast<const uint32_t*>(&h2);
            }
            // PV of the previous block must be done: P buffer free, O current.
            if (!__all_sync(0xffffffffu, tc::mbar_wait(bar(B_PEMPTY), (uint32_t(j) & 1u) ^ 1u, s_abort, P.err,
                                                       kErrWaitSoftmax))) {
                ok = false;
                break;
            }
            tc::tc_fence_after();
            if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
                for (int q = 0; q < D / 32; ++q) {
                    float v[32];
                    const uint32_t ta = tmem + lane_base + C::COL_O + q * 32;
                    tc::tmem_ld32(ta, v);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= rescale ? alpha : 1.f;
                    tc::tmem_st32(ta, v);
                }
                tc::tmem_wait_st();
            }
            l_run = l_run * alpha + lsum;
            // P row -> smem (K-major over keys, 128-byte swizzle)
#pragma unroll
            for (int cc = 0; cc < C::BN / 8; ++cc) {
                const uint4 v = make_uint4(pk[4 * cc], pk[4 * cc + 1], pk[4 * cc + 2], pk[4 * cc + 3]);
                *reinterpret_cast<uint4*>(p_s + (cc / 8) * (kRows * 128) + row * 128 + (((cc % 8) ^ (row % 8)) * 16)) = v;
            }
            tc::fence_proxy_async_smem();
            tc::tc_fence_before();
            tc::mbar_arrive(bar(B_PFULL));
        }
        // ---- epilogue: partial state of this row ----
        if (ok && nblk > 0 &&
            __all_sync(0xffffffffu, tc::mbar_wait(bar(B_ODONE), 0, s_abort, P.err, kErrWaitSoftmax))) {
            tc::tc_fence_after();
            const size_t idx = size_t(split) * P.B * P.Hq + size_t(out_row);
            float* op = P.ws_o + idx * D;
#pragma unroll
            for (int q = 0; q < D / 32; ++q) {
                float v[32];
                tc::tmem_ld32(tmem + lane_base + C::COL_O + q * 32, v);
                tc::tmem_wait_ld();
                if (valid) {
#pragma unroll
                    for (int i = 0; i < 32; i += 4)
                        *reinterpret_cast<float4*>(op + q * 32 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                }
            }
            if (valid) P.ws_ml[idx] = make_float2(m_run, l_run);
        } else if (nblk == 0 && valid) {
            const size_t idx = size_t(split) * P.B * P.Hq + size_t(out_row);
            P.ws_ml[idx] = make_float2(-INFINITY, 0.f);
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
    TcParams tp{p, nsplit, split_keys};
    const dim3 grid(unsigned(p.n_tiles * p.Hkv * nsplit)), block(kThreads);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.D) {
        case 64: {
            static bool attr = false;
            if (!attr) {
                cudaFuncSetAttribute(prefix_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<64>::SMEM);
                attr = true;
            }
            prefix_tc_kernel<64><<<grid, block, Cfg<64>::SMEM, st>>>(m[0], m[1], m[2], m[3], tp);
            break;
        }
        case 128: {
            static bool attr = false;
            if (!attr) {
                cudaFuncSetAttribute(prefix_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     Cfg<128>::SMEM);
                attr = true;
            }
            prefix_tc_kernel<128><<<grid, block, Cfg<128>::SMEM, st>>>(m[0], m[1], m[2], m[3], tp);
            break;
        }
        case 256: {
            static bool attr = false;
            if (!attr) {
                cudaFuncSetAttribute(prefix_tc_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     Cfg<256>::SMEM);
                attr = true;
            }
            prefix_tc_kernel<256><<<grid, block, Cfg<256>::SMEM, st>>>(m[0], m[1], m[2], m[3], tp);
            break;
        }
        default: return int(cudaErrorInvalidValue);
    }
    return int(cudaGetLastError());
}

}  // namespace splice
