// C ABI of the spliced decode-attention library (include/splice.h):
// argument validation, descriptor lifetime, device tables, and the launch
// sequence of one decode step.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "splice_internal.h"

using splice::AttnParams;
using splice::Plan;

struct splice_desc {
    bool on_device = false;
    splice_model_shape shape{};
    int P = 0, Tp = 0, Dslots = 0, Dst = 0, B = 0, T = 0;
    std::vector<int32_t> slot_stored;   // [Dslots] stored-donor index or -1
    std::vector<splice_donor_kind> kinds;
    std::vector<splice_seq> seqs;
    Plan plan;
    int device = -1;
    int sms = 0;                        // multiprocessors of the device
    int pass_order = 0;                 // 0 chosen per call, 1 prompt-span pass first, 2 generated-span pass first
    // Device tables, one allocation.
    char* dev = nullptr;
    std::vector<char> staging;          // host image of `dev`, kept for the async upload
    uint8_t* d_src = nullptr;
    int32_t* d_seq_prompt = nullptr;
    int32_t* d_seq_slot = nullptr;
    int32_t* d_slot_stored = nullptr;
    int32_t* d_tiles = nullptr;
    int32_t* d_group_prompt = nullptr;
    int32_t* d_group_src = nullptr;
    int32_t* d_group_seqs = nullptr;
    int32_t* d_group_mask = nullptr;
    int32_t* d_slot_delta = nullptr;
    unsigned* d_err = nullptr;
    unsigned* d_sched = nullptr;   // [8] work counters, finished counts and the completion flag of the passes
    // Measurement: launch counter and optional per-launch event timing.
    long long launches = 0;
    bool profiling = false;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> events[SPLICE_KERNEL_KINDS];
    size_t events_used[SPLICE_KERNEL_KINDS] = {0, 0, 0, 0};
    // Delta mode: which slots are read through their delta encoding, the
    // caller's delta buffer, and the largest encoded count of those slots.
    std::vector<uint8_t> slot_delta;    // [Dslots]
    bool delta_on = false;
    char* delta = nullptr;
    int delta_max = 0;
    // TMA tensor maps of the clean and donor stores and of the delta rows
    // (K, V each), rebuilt when the store pointers change.
    alignas(64) unsigned char maps[6][128] = {};
    const void* map_ptr[6] = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
};

namespace {

thread_local std::string g_last_error;

splice_status fail(splice_status st, const char* f, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, f);
    std::vsnprintf(buf, sizeof buf, f, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

splice_status cuda_fail(cudaError_t e, const char* what) {
    return fail(SPLICE_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Restores the caller's current device on scope exit.
struct DeviceGuard {
    int prev = -1;
    bool changed = false;
    cudaError_t err = cudaSuccess;
    explicit DeviceGuard(int dev) {
        err = cudaGetDevice(&prev);
        if (err == cudaSuccess && prev != dev) {
            err = cudaSetDevice(dev);
            changed = err == cudaSuccess;
        }
    }
    ~DeviceGuard() {
        if (changed) cudaSetDevice(prev);
    }
};

splice_status validate_create(const splice_model_shape* sh, int P, int Tp, int Dslots,
                              const splice_donor_kind* kinds, int B, const splice_seq* seqs,
                              int T, splice_desc** out) {
    if (!out) return fail(SPLICE_EINVAL, "out is NULL");
    *out = nullptr;
    if (!sh) return fail(SPLICE_EINVAL, "shape is NULL");
    if (sh->num_layers < 1) return fail(SPLICE_EINVAL, "num_layers %d < 1", sh->num_layers);
    if (sh->num_kv_heads < 1 || sh->num_q_heads < sh->num_kv_heads ||
        sh->num_q_heads % sh->num_kv_heads != 0)
        return fail(SPLICE_EINVAL, "num_q_heads %d must be a positive multiple of num_kv_heads %d",
                    sh->num_q_heads, sh->num_kv_heads);
    if (sh->num_q_heads / sh->num_kv_heads > 16)
        return fail(SPLICE_EINVAL, "group size %d > 16", sh->num_q_heads / sh->num_kv_heads);
    if (sh->head_dim != 64 && sh->head_dim != 128 && sh->head_dim != 256)
        return fail(SPLICE_EINVAL, "head_dim %d not in {64, 128, 256}", sh->head_dim);
    if (sh->sliding_window < 0 || sh->global_every < 0)
        return fail(SPLICE_EINVAL, "negative sliding_window or global_every");
    if (!std::isfinite(sh->sm_scale)) return fail(SPLICE_EINVAL, "sm_scale is not finite");
    if (P < 1 || Tp < 1 || B < 1 || T < 1)
        return fail(SPLICE_EINVAL, "num_prompts, prompt_len, num_seqs and max_steps must be >= 1");
    if (Dslots < 1 || Dslots > 250) return fail(SPLICE_EINVAL, "num_donor_slots %d not in [1, 250]", Dslots);
    if (!kinds || !seqs) return fail(SPLICE_EINVAL, "slot_kinds or seqs is NULL");
    int dst = 0;
    for (int k = 0; k < Dslots; ++k) {
        if (int(kinds[k]) < 0 || int(kinds[k]) > 4)
            return fail(SPLICE_EINVAL, "slot %d has unknown donor kind %d", k, int(kinds[k]));
        if (kinds[k] != SPLICE_DONOR_ZERO) ++dst;
    }
    for (int s = 0; s < B; ++s) {
        const splice_seq& q = seqs[s];
        if (q.prompt_id < 0 || q.prompt_id >= P)
            return fail(SPLICE_EINVAL, "seq %d: prompt_id %d out of range", s, q.prompt_id);
        if (q.donor_slot < 0 || q.donor_slot >= Dslots)
            return fail(SPLICE_EINVAL, "seq %d: donor_slot %d out of range", s, q.donor_slot);
        if (q.L < 0 || q.W < 0) return fail(SPLICE_EINVAL, "seq %d: negative L or W", s);
    }
    const long long rows = 1LL * P * sh->num_layers * sh->num_kv_heads * Tp;
    if (rows >= (1LL << 31) || rows * std::max(dst, 1) >= (1LL << 31))
        return fail(SPLICE_EINVAL, "prompt stores exceed 2^31 rows");
    return SPLICE_OK;
}

splice_status create_common(const splice_model_shape* sh, int P, int Tp, int Dslots,
                            const splice_donor_kind* kinds, int B, const splice_seq* seqs, int T,
                            splice_desc** out, splice_desc*& d) {
    splice_status st = validate_create(sh, P, Tp, Dslots, kinds, B, seqs, T, out);
    if (st != SPLICE_OK) return st;
    d = new (std::nothrow) splice_desc();
    if (!d) return fail(SPLICE_ENOMEM, "descriptor allocation failed");
    try {
        d->shape = *sh;
        d->P = P;
        d->Tp = Tp;
        d->Dslots = Dslots;
        d->B = B;
        d->T = T;
        d->seqs.assign(seqs, seqs + B);
        d->kinds.assign(kinds, kinds + Dslots);
        d->slot_delta.assign(Dslots, 0);
        d->slot_stored.assign(Dslots, -1);
        for (int k = 0; k < Dslots; ++k)
            if (kinds[k] != SPLICE_DONOR_ZERO) d->slot_stored[k] = d->Dst++;
        std::string e = splice::build_plan(*sh, P, Tp, Dslots, kinds, B, seqs, T, nullptr, d->plan);
        if (!e.empty()) {
            delete d;
            d = nullptr;
            return fail(SPLICE_EINVAL, "%s", e.c_str());
        }
    } catch (const std::bad_alloc&) {
        delete d;
        d = nullptr;
        return fail(SPLICE_ENOMEM, "host allocation failed while planning");
    }
    return SPLICE_OK;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// (Re)builds the device table block of a descriptor from its host plan and
// copies it on `stream`; frees the previous block (no launch that uses it may
// be in flight).  The error word and the work counter start at zero.
splice_status upload_tables(splice_desc* d, void* stream) {
    const Plan& pl = d->plan;
    struct Part {
        const void* src;
        size_t bytes;
        size_t off;
    };
    std::vector<int32_t> seq_prompt(d->B), seq_slot(d->B), slot_delta(d->Dslots);
    for (int s = 0; s < d->B; ++s) {
        seq_prompt[s] = d->seqs[s].prompt_id;
        seq_slot[s] = d->seqs[s].donor_slot;
    }
    for (int k = 0; k < d->Dslots; ++k) slot_delta[k] = d->slot_delta[k] ? 1 : 0;
    const unsigned zero = 0;
    const unsigned sched_zero[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    Part parts[] = {
        {pl.src.data(), pl.src.size(), 0},
        {seq_prompt.data(), seq_prompt.size() * 4, 0},
        {seq_slot.data(), seq_slot.size() * 4, 0},
        {d->slot_stored.data(), d->slot_stored.size() * 4, 0},
        {pl.tiles.data(), pl.tiles.size() * 4, 0},
        {pl.group_prompt.data(), pl.group_prompt.size() * 4, 0},
        {pl.group_src.data(), pl.group_src.size() * 4, 0},
        {pl.group_seqs.data(), pl.group_seqs.size() * 4, 0},
        {&zero, sizeof zero, 0},
        {sched_zero, sizeof sched_zero, 0},
        {pl.group_mask.data(), pl.group_mask.size() * 4, 0},
        {slot_delta.data(), slot_delta.size() * 4, 0},
    };
    size_t total = 0;
    for (Part& p : parts) {
        p.off = total;
        total = align_up(total + std::max<size_t>(p.bytes, 4), 256);
    }
    try {
        d->staging.assign(total, 0);
    } catch (const std::bad_alloc&) {
        return fail(SPLICE_ENOMEM, "host staging allocation failed");
    }
    for (const Part& p : parts)
        if (p.bytes) std::memcpy(d->staging.data() + p.off, p.src, p.bytes);
    char* b = nullptr;
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(&b), total);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return e == cudaErrorMemoryAllocation ? fail(SPLICE_ENOMEM, "cudaMalloc of %zu bytes failed", total)
                                              : cuda_fail(e, "cudaMalloc");
    }
    e = cudaMemcpyAsync(b, d->staging.data(), total, cudaMemcpyHostToDevice, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) {
        cudaFree(b);
        return cuda_fail(e, "cudaMemcpyAsync of descriptor tables");
    }
    if (d->dev) {
        e = cudaFree(d->dev);
        if (e != cudaSuccess) {
            cudaFree(b);
            return cuda_fail(e, "cudaFree of the previous descriptor tables");
        }
    }
    d->dev = b;
    d->d_src = reinterpret_cast<uint8_t*>(b + parts[0].off);
    d->d_seq_prompt = reinterpret_cast<int32_t*>(b + parts[1].off);
    d->d_seq_slot = reinterpret_cast<int32_t*>(b + parts[2].off);
    d->d_slot_stored = reinterpret_cast<int32_t*>(b + parts[3].off);
    d->d_tiles = reinterpret_cast<int32_t*>(b + parts[4].off);
    d->d_group_prompt = reinterpret_cast<int32_t*>(b + parts[5].off);
    d->d_group_src = reinterpret_cast<int32_t*>(b + parts[6].off);
    d->d_group_seqs = reinterpret_cast<int32_t*>(b + parts[7].off);
    d->d_err = reinterpret_cast<unsigned*>(b + parts[8].off);
    d->d_sched = reinterpret_cast<unsigned*>(b + parts[9].off);
    d->d_group_mask = reinterpret_cast<int32_t*>(b + parts[10].off);
    d->d_slot_delta = reinterpret_cast<int32_t*>(b + parts[11].off);
    return SPLICE_OK;
}

// Layout of the caller's delta buffer (include/splice.h, splice_delta_bytes).
struct DeltaLayout {
    size_t spans = 0, mask_off = 0, count_off = 0, k_off = 0, v_off = 0, total = 0;
    int w32 = 0;
};

DeltaLayout delta_layout(const splice_desc* d) {
    DeltaLayout L;
    if (d->Dst == 0) return L;
    const splice_model_shape& sh = d->shape;
    L.spans = size_t(d->P) * d->Dst * sh.num_layers * sh.num_kv_heads;
    L.w32 = 4 * ((d->Tp + 127) / 128);     // whole 128-key blocks: a tile's last block stays inside
    const size_t rows = L.spans * size_t(d->Tp) * size_t(sh.head_dim) * 2;
    L.mask_off = 0;
    L.count_off = align_up(L.spans * size_t(L.w32) * 4, 256);
    L.k_off = align_up(L.count_off + L.spans * 4, 256);
    L.v_off = align_up(L.k_off + rows, 256);
    L.total = L.v_off + rows;
    return L;
}

// Rebuilds the plan for the descriptor's current slot_delta.
splice_status replan(splice_desc* d) {
    try {
        std::string e = splice::build_plan(d->shape, d->P, d->Tp, d->Dslots, d->kinds.data(), d->B, d->seqs.data(), d->T,
                                           d->slot_delta.data(), d->plan);
        if (!e.empty()) return fail(SPLICE_EINVAL, "%s", e.c_str());
    } catch (const std::bad_alloc&) {
        return fail(SPLICE_ENOMEM, "host allocation failed while planning");
    }
    return SPLICE_OK;
}


// Runs one kernel launcher, counting it and, when profiling, bracketing it
// with a pair of events on its stream.
template <class F>
cudaError_t timed_launch(splice_desc* d, int kind, void* stream, F&& launch) {
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    std::pair<cudaEvent_t, cudaEvent_t>* ev = nullptr;
    if (d->profiling) {
        auto& pool = d->events[kind];
        if (d->events_used[kind] == pool.size()) {
            cudaEvent_t a, b;
            cudaError_t e = cudaEventCreate(&a);
            if (e != cudaSuccess) return e;
            e = cudaEventCreate(&b);
            if (e != cudaSuccess) {
                cudaEventDestroy(a);
                return e;
            }
            pool.emplace_back(a, b);
        }
        ev = &pool[d->events_used[kind]++];
        cudaError_t e = cudaEventRecord(ev->first, st);
        if (e != cudaSuccess) return e;
    }
    cudaError_t e = cudaError_t(launch());
    if (e != cudaSuccess) return e;
    ++d->launches;
    if (ev) e = cudaEventRecord(ev->second, st);
    return e;
}

// The workspace: (m, l) of every partial state, then o, each part starting
// on a 256-byte boundary whatever the alignment of the caller's pointer (the
// kernels store o with 32-byte vector stores), hence the 256 bytes of slack.
size_t workspace_bytes_of(const splice_desc* d) {
    const size_t rows = size_t(d->B) * d->shape.num_q_heads;
    const size_t ml = align_up(size_t(splice::kMaxSplits) * rows * sizeof(float2), 256);
    const size_t o = size_t(splice::kMaxSplits) * rows * d->shape.head_dim * sizeof(float);
    return 256 + ml + o;
}

// One attention call: validation, the (epoch, layer class) table of (layer,
// step), and the launches of the generated-span pass, the prompt-span pass
// and the merge.  k_new / v_new non-NULL: the generated-span pass also
// appends them at entry step - 1 (the fused decode step).
splice_status attn_common(splice_desc* d, int layer, int step, const splice_bf16* q, const splice_bf16* k_new,
                          const splice_bf16* v_new, const splice_bf16* k_clean, const splice_bf16* v_clean,
                          const splice_bf16* k_donor, const splice_bf16* v_donor, splice_bf16* k_suffix,
                          splice_bf16* v_suffix, float* out, void* workspace, size_t workspace_bytes, void* stream,
                          const char* who) {
    if (!d) return fail(SPLICE_EINVAL, "%s: descriptor is NULL", who);
    if (!d->on_device) return fail(SPLICE_ESTATE, "%s: host-only descriptor", who);
    if (layer < 0 || layer >= d->shape.num_layers) return fail(SPLICE_EINVAL, "%s: layer %d out of range", who, layer);
    if (step < 0 || step > d->T) return fail(SPLICE_EINVAL, "%s: step %d not in [0, %d]", who, step, d->T);
    if (!q || !k_clean || !v_clean || !out || !workspace)
        return fail(SPLICE_EINVAL, "%s: NULL tensor or workspace", who);
    if (step > 0 && (!k_suffix || !v_suffix)) return fail(SPLICE_EINVAL, "%s: NULL generated-span store", who);
    if (d->Dst > 0 && (!k_donor || !v_donor)) return fail(SPLICE_EINVAL, "%s: NULL donor store", who);
    const void* ptrs[] = {q, k_new, v_new, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix, out, workspace};
    for (const void* p : ptrs)
        if (p && !aligned16(p)) return fail(SPLICE_EINVAL, "%s: tensor not 16-byte aligned", who);
    if (workspace_bytes < workspace_bytes_of(d))
        return fail(SPLICE_EINVAL, "%s: workspace of %zu bytes < %zu", who, workspace_bytes, workspace_bytes_of(d));
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "earlier CUDA error");

    const splice_model_shape& sh = d->shape;
    const int tab = d->plan.table_of(layer, step);
    const splice::Visible vis = splice::visible_keys(sh, d->Tp, layer, step);
    const size_t rows = size_t(d->B) * sh.num_q_heads;
    AttnParams p{};
    p.q = q;
    p.kc = k_clean;
    p.vc = v_clean;
    p.kd = k_donor;
    p.vd = v_donor;
    p.ks = k_suffix;
    p.vs = v_suffix;
    p.kn = k_new;
    p.vn = v_new;
    p.ks_w = k_suffix;
    p.vs_w = v_suffix;
    p.fuse_append = k_new ? 1 : 0;
    p.out = out;
    char* ws_base = reinterpret_cast<char*>(align_up(reinterpret_cast<uintptr_t>(workspace), 256));
    p.ws_ml = reinterpret_cast<float2*>(ws_base);
    p.ws_o = reinterpret_cast<float*>(ws_base + align_up(size_t(splice::kMaxSplits) * rows * sizeof(float2), 256));
    p.src = d->d_src + size_t(tab) * d->B;
    p.seq_prompt = d->d_seq_prompt;
    p.seq_slot = d->d_seq_slot;
    p.slot_stored = d->d_slot_stored;
    p.tiles = d->d_tiles + 4 * size_t(d->plan.table_tile_off[tab]);
    p.n_tiles = d->plan.table_tile_off[tab + 1] - d->plan.table_tile_off[tab];
    p.group_prompt = d->d_group_prompt;
    p.group_src = d->d_group_src;
    p.group_seqs = d->d_group_seqs;
    p.err = d->d_err;
    p.sched = d->d_sched;
    p.B = d->B;
    p.N = sh.num_layers;
    p.Hq = sh.num_q_heads;
    p.Hkv = sh.num_kv_heads;
    p.D = sh.head_dim;
    p.G = sh.num_q_heads / sh.num_kv_heads;
    p.Tp = d->Tp;
    p.T = d->T;
    p.Dst = d->Dst;
    p.layer = layer;
    p.step = step;
    p.p_lo = vis.p_lo;
    p.p_hi = vis.p_hi;
    p.s_lo = vis.s_lo;
    p.s_hi = vis.s_hi;
    const int p_vis = vis.p_hi - vis.p_lo, s_vis = vis.s_hi - vis.s_lo;
    // In delta mode a delta row's span splits and delta-row splits share the
    // kMaxPrefixSplits prompt-span partial slots.
    const int max_splits = d->delta_on ? splice::kMaxPrefixSplits / 2 : splice::kMaxPrefixSplits;
    int tc_split = 0, tc_keys = 0;
    int bounds[splice::kMaxPrefixSplits + 1] = {0};
    if (p_vis > 0) {
        tc_split = splice::prefix_tc_splits(sh.head_dim, p_vis, max_splits, bounds);
        tc_keys = bounds[1];           // the longest split
    }
    p.nsp = tc_split;
    p.n_span_tiles = d->plan.table_span_tiles[tab];
    p.group_mask = d->d_group_mask;
    p.slot_delta = d->d_slot_delta;
    p.delta_on = d->delta_on ? 1 : 0;
    p.nsd = 0;
    if (d->delta_on) {
        const DeltaLayout dl = delta_layout(d);
        p.dmask = reinterpret_cast<const uint32_t*>(d->delta + dl.mask_off);
        p.dcount = reinterpret_cast<const int32_t*>(d->delta + dl.count_off);
        p.delta_w32 = dl.w32;
        if (tc_keys > 0) p.nsd = std::min(max_splits, (d->delta_max + tc_keys - 1) / tc_keys);
    }
    {
        // Generated-span items: (sequence, kv head, row chunk, key split).
        // Split so every resident warp gets about two items, but keep at
        // least 64 keys per split.  Every split costs a partial state to
        // write and merge; the prompt-span pass queued behind this one fills
        // the SMs its last warps leave idle, so few splits pay off even
        // where the items do not share out evenly over the warps.
        const int G = sh.num_q_heads / sh.num_kv_heads;
        const int gt = G % 4 == 0 ? 4 : (G % 2 == 0 ? 2 : 1);
        const long base_items = long(d->B) * sh.num_kv_heads * (G / gt);
        const long want = 2L * splice::generated_span_resident_warps(sh.head_dim);
        int ns = int(std::min<long>(splice::kMaxSuffixSplits, std::max<long>(1, (want + base_items - 1) / base_items)));
        ns = std::min(ns, std::max(1, s_vis / 64));
        p.nss = s_vis > 0 ? ns : 0;
    }
    p.p_chunk = tc_keys;
    p.s_chunk = p.nss ? (s_vis + p.nss - 1) / p.nss : 0;
    p.scale_log2 = sh.sm_scale * 1.4426950408889634f;

    // The two passes read disjoint inputs and write disjoint partial slots,
    // and run as programmatic dependent launches: the call's first pass
    // waits for whatever precedes it on the stream before it reads anything,
    // then lets the second pass launch; the second pass's CTAs take the SMs
    // the first pass's CTAs leave, and it waits for the first pass before it
    // exits; the merge is queued behind the second pass (unless the
    // generated-span pass merges every row, p.gs_merge below).  So the first pass's
    // tail is filled and the second pass's is not.  The generated-span pass
    // goes first when the prompt-span pass holds at least
    // kPrefixFirstKeysPerSm keys per SM: then the prompt-span pass's items
    // fill the generated-span pass's tail.  A smaller prompt-span pass goes
    // first: its short run and its tail (part of the SMs idle while its last
    // items finish) are filled by the generated-span pass's run-time claimed
    // items.  So does a prompt-span pass with more than
    // kPrefixFirstGenRatio times the generated-span pass's keys (x row
    // chunks): the generated-span pass's short items then fill its tail.
    // With per-launch timing on, the events between the launches serialise
    // everything.
    const bool gs_work = p.nss > 0;
    const long prefix_items = long(p.n_span_tiles) * sh.num_kv_heads * p.nsp +
                              long(p.n_tiles - p.n_span_tiles) * sh.num_kv_heads * p.nsd;
    const bool prefix_launched = p.nsp > 0 && prefix_items > 0;
    const int box = splice::prefix_tc_box_rows(sh.head_dim);
    const long prefix_keys =
        (long(p.n_span_tiles) * ((p_vis + box - 1) / box) +
         long(p.n_tiles - p.n_span_tiles) * (p.nsd ? (d->delta_max + box - 1) / box : 0)) *
        sh.num_kv_heads * box;
    const long gs_keys = long(d->B) * sh.num_kv_heads * (p.G / (p.G % 4 == 0 ? 4 : (p.G % 2 == 0 ? 2 : 1))) * s_vis;
    const bool prefix_first =
        prefix_launched &&
        (d->pass_order == 1 ||
         (d->pass_order == 0 && (prefix_keys < long(d->sms) * splice::kPrefixFirstKeysPerSm ||
                                 gs_keys * splice::kPrefixFirstGenRatio < prefix_keys)));
    p.gs_after_prefix = gs_work && prefix_launched && prefix_first && !d->profiling ? 1 : 0;
    p.prefix_after_gs = gs_work && prefix_launched && !prefix_first && !d->profiling ? 1 : 0;
    // Behind the prompt-span pass, with one prompt-span and one
    // generated-span split per row and no delta rows, the generated-span
    // pass merges every row itself and writes the output: ZERO rows at the
    // item's end, the others there once the prompt-span pass has completed
    // (a flag it reads without waiting), else at the warp's end after the
    // grid dependency wait.  No merge kernel is launched then.
    p.gs_merge = p.gs_after_prefix && p.nss == 1 && p.nsp == 1 && !p.delta_on &&
                         splice::generated_span_can_merge(sh.head_dim, p.G)
                     ? 1
                     : 0;
    auto launch_prefix = [&]() -> splice_status {
        // Tensor maps over the stores viewed as [rows][d]; the delta rows
        // have the donor store's layout.
        const long rows_c = long(d->P) * sh.num_layers * sh.num_kv_heads * d->Tp;
        const long rows_d = d->Dst ? rows_c * d->Dst : rows_c;
        const DeltaLayout dl = delta_layout(d);
        const void* xk = d->delta_on ? static_cast<const void*>(d->delta + dl.k_off) : k_clean;
        const void* xv = d->delta_on ? static_cast<const void*>(d->delta + dl.v_off) : v_clean;
        const void* mp[6] = {k_clean, v_clean, d->Dst ? k_donor : k_clean, d->Dst ? v_donor : v_clean, xk, xv};
        const long mrows[6] = {rows_c, rows_c, rows_d, rows_d, d->delta_on ? rows_d : rows_c,
                               d->delta_on ? rows_d : rows_c};
        for (int i = 0; i < 6; ++i) {
            if (d->map_ptr[i] == mp[i]) continue;
            if (splice::make_kv_tensor_map(d->maps[i], mp[i], mrows[i], sh.head_dim, box) != 0)
                return fail(SPLICE_ECUDA, "cuTensorMapEncodeTiled failed for store %d", i);
            d->map_ptr[i] = mp[i];
        }
        const cudaError_t le = timed_launch(d, 1, stream, [&] {
            return splice::launch_prefix_tc(p, d->maps, bounds, tc_keys, stream, !d->profiling);
        });
        if (le != cudaSuccess) return cuda_fail(le, "prompt-span tensor-core pass launch");
        return SPLICE_OK;
    };
    auto launch_gs = [&]() -> splice_status {
        const cudaError_t le =
            timed_launch(d, 2, stream, [&] { return splice::launch_generated_span(p, stream, !d->profiling); });
        if (le != cudaSuccess) return cuda_fail(le, "generated-span partials launch");
        return SPLICE_OK;
    };
    if (prefix_launched && prefix_first) {
        const splice_status st = launch_prefix();
        if (st != SPLICE_OK) return st;
    }
    if (gs_work) {
        const splice_status st = launch_gs();
        if (st != SPLICE_OK) return st;
    }
    if (prefix_launched && !prefix_first) {
        const splice_status st = launch_prefix();
        if (st != SPLICE_OK) return st;
    }
    if (p.gs_merge) return SPLICE_OK;
    const bool merge_overlap = (prefix_launched || gs_work) && !d->profiling;
    e = timed_launch(d, 3, stream, [&] { return splice::launch_merge(p, stream, merge_overlap); });
    if (e != cudaSuccess) return cuda_fail(e, "merge launch");
    return SPLICE_OK;
}

}  // namespace

void splice::set_last_error(const char* msg) { g_last_error = msg; }

int splice::desc_device(const splice_desc* d) { return d && d->on_device ? d->device : -1; }

extern "C" {

const char* splice_status_str(splice_status s) {
    switch (s) {
        case SPLICE_OK: return "ok";
        case SPLICE_EINVAL: return "invalid argument";
        case SPLICE_ENOMEM: return "out of memory";
        case SPLICE_ECUDA: return "CUDA error";
        case SPLICE_ESTATE: return "descriptor state does not allow this call";
        case SPLICE_EDEVICE: return "kernel-side error";
    }
    return "unknown status";
}

const char* splice_last_error(void) { return g_last_error.c_str(); }

splice_status splice_desc_create_host(const splice_model_shape* sh, int P, int Tp, int Dslots,
                                       const splice_donor_kind* kinds, int B, const splice_seq* seqs,
                                       int T, splice_desc** out) {
    splice_desc* d = nullptr;
    splice_status st = create_common(sh, P, Tp, Dslots, kinds, B, seqs, T, out, d);
    if (st != SPLICE_OK) return st;
    *out = d;
    return SPLICE_OK;
}

splice_status splice_desc_create(const splice_model_shape* sh, int P, int Tp, int Dslots,
                                  const splice_donor_kind* kinds, int B, const splice_seq* seqs,
                                  int T, void* stream, splice_desc** out) {
    splice_desc* d = nullptr;
    splice_status st = create_common(sh, P, Tp, Dslots, kinds, B, seqs, T, out, d);
    if (st != SPLICE_OK) return st;
    cudaError_t e = cudaGetDevice(&d->device);
    if (e != cudaSuccess) {
        delete d;
        return cuda_fail(e, "cudaGetDevice");
    }
    e = cudaDeviceGetAttribute(&d->sms, cudaDevAttrMultiProcessorCount, d->device);
    if (e != cudaSuccess) {
        delete d;
        return cuda_fail(e, "cudaDeviceGetAttribute");
    }
    st = upload_tables(d, stream);
    if (st != SPLICE_OK) {
        delete d;
        return st;
    }
    d->on_device = true;
    *out = d;
    return SPLICE_OK;
}

splice_status splice_desc_destroy(splice_desc* d) {
    if (!d) return SPLICE_OK;
    splice_status st = SPLICE_OK;
    if (d->dev) {
        DeviceGuard g(d->device);
        for (auto& pool : d->events)
            for (auto& ev : pool) {
                cudaEventDestroy(ev.first);
                cudaEventDestroy(ev.second);
            }
        cudaError_t e = cudaFree(d->dev);
        if (e != cudaSuccess) st = cuda_fail(e, "cudaFree of descriptor tables");
    }
    delete d;
    return st;
}

size_t splice_workspace_bytes(const splice_desc* d) { return d ? workspace_bytes_of(d) : 0; }

int splice_num_stored_donor_slots(const splice_desc* d) { return d ? d->Dst : -1; }

splice_status suffix_kv_append(splice_desc* d, int layer, int step, const splice_bf16* k_new,
                               const splice_bf16* v_new, splice_bf16* k_suffix,
                               splice_bf16* v_suffix, void* stream) {
    if (!d) return fail(SPLICE_EINVAL, "descriptor is NULL");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    if (layer < 0 || layer >= d->shape.num_layers) return fail(SPLICE_EINVAL, "layer %d out of range", layer);
    if (step < 1 || step > d->T) return fail(SPLICE_EINVAL, "append step %d not in [1, %d]", step, d->T);
    if (!k_new || !v_new || !k_suffix || !v_suffix) return fail(SPLICE_EINVAL, "NULL tensor");
    if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_suffix) || !aligned16(v_suffix))
        return fail(SPLICE_EINVAL, "tensor not 16-byte aligned");
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "earlier CUDA error");
    e = timed_launch(d, 0, stream, [&] {
        return splice::launch_append(k_new, v_new, k_suffix, v_suffix, d->B, d->shape.num_layers,
                                     d->shape.num_kv_heads, d->shape.head_dim, d->T, layer, step, stream);
    });
    if (e != cudaSuccess) return cuda_fail(e, "append launch");
    return SPLICE_OK;
}

splice_status spliced_decode_attn(splice_desc* d, int layer, int step, const splice_bf16* q,
                                  const splice_bf16* k_clean, const splice_bf16* v_clean,
                                  const splice_bf16* k_donor, const splice_bf16* v_donor,
                                  const splice_bf16* k_suffix, const splice_bf16* v_suffix, float* out,
                                  void* workspace, size_t workspace_bytes, void* stream) {
    return attn_common(d, layer, step, q, nullptr, nullptr, k_clean, v_clean, k_donor, v_donor,
                       const_cast<splice_bf16*>(k_suffix), const_cast<splice_bf16*>(v_suffix), out, workspace,
                       workspace_bytes, stream, "spliced_decode_attn");
}

splice_status spliced_decode_step(splice_desc* d, int layer, int step, const splice_bf16* q,
                                  const splice_bf16* k_new, const splice_bf16* v_new,
                                  const splice_bf16* k_clean, const splice_bf16* v_clean,
                                  const splice_bf16* k_donor, const splice_bf16* v_donor, splice_bf16* k_suffix,
                                  splice_bf16* v_suffix, float* out, void* workspace, size_t workspace_bytes,
                                  void* stream) {
    if (d && (step < 1 || step > d->T))
        return fail(SPLICE_EINVAL, "spliced_decode_step: step %d not in [1, %d]", step, d->T);
    if (!k_new || !v_new) return fail(SPLICE_EINVAL, "spliced_decode_step: NULL k_new or v_new");
    return attn_common(d, layer, step, q, k_new, v_new, k_clean, v_clean, k_donor, v_donor, k_suffix, v_suffix,
                       out, workspace, workspace_bytes, stream, "spliced_decode_step");
}

size_t splice_delta_bytes(const splice_desc* d) { return d ? delta_layout(d).total : 0; }

splice_status splice_delta_build(splice_desc* d, const splice_bf16* k_clean, const splice_bf16* v_clean,
                                 const splice_bf16* k_donor, const splice_bf16* v_donor, void* delta,
                                 size_t delta_bytes, float max_fraction, float* slot_fraction, void* stream) {
    if (!d) return fail(SPLICE_EINVAL, "descriptor is NULL");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    if (d->Dst == 0) return fail(SPLICE_EINVAL, "the descriptor has no stored donor slot");
    if (d->shape.sliding_window > 0)
        return fail(SPLICE_EINVAL, "delta encoding needs a descriptor without a sliding window");
    if (!(max_fraction >= 0.f && max_fraction <= 1.f)) return fail(SPLICE_EINVAL, "max_fraction not in [0, 1]");
    if (!k_clean || !v_clean || !k_donor || !v_donor || !delta) return fail(SPLICE_EINVAL, "NULL tensor or buffer");
    const void* ptrs[] = {k_clean, v_clean, k_donor, v_donor, delta};
    for (const void* p : ptrs)
        if (!aligned16(p)) return fail(SPLICE_EINVAL, "tensor not 16-byte aligned");
    const DeltaLayout dl = delta_layout(d);
    if (delta_bytes < dl.total) return fail(SPLICE_EINVAL, "delta buffer of %zu bytes < %zu", delta_bytes, dl.total);
    if (size_t(dl.w32) * 8 > 200 * 1024) return fail(SPLICE_EINVAL, "prompt_len %d too long for delta encoding", d->Tp);
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "earlier CUDA error");
    const splice_model_shape& sh = d->shape;
    char* b = static_cast<char*>(delta);
    e = cudaError_t(splice::launch_delta_build(
        k_clean, v_clean, k_donor, v_donor, reinterpret_cast<uint32_t*>(b + dl.mask_off),
        reinterpret_cast<int32_t*>(b + dl.count_off), reinterpret_cast<uint16_t*>(b + dl.k_off),
        reinterpret_cast<uint16_t*>(b + dl.v_off), d->P, d->Dst, sh.num_layers, sh.num_kv_heads, d->Tp, sh.head_dim,
        dl.w32, stream));
    if (e != cudaSuccess) return cuda_fail(e, "delta encoding launch");
    std::vector<int32_t> counts;
    try {
        counts.resize(dl.spans);
    } catch (const std::bad_alloc&) {
        return fail(SPLICE_ENOMEM, "host allocation failed");
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    e = cudaMemcpyAsync(counts.data(), b + dl.count_off, dl.spans * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "reading the delta counts");
    // per stored slot: encoded rows / rows of its spans
    const size_t per_slot = size_t(sh.num_layers) * sh.num_kv_heads;
    std::vector<double> frac(d->Dst, 0.0);
    std::vector<int> maxc(d->Dst, 0);
    for (int p = 0; p < d->P; ++p)
        for (int stq = 0; stq < d->Dst; ++stq)
            for (size_t i = 0; i < per_slot; ++i) {
                const int c = counts[(size_t(p) * d->Dst + stq) * per_slot + i];
                frac[stq] += c;
                maxc[stq] = std::max(maxc[stq], c);
            }
    const double rows_per_slot = double(d->P) * double(per_slot) * double(d->Tp);
    std::vector<uint8_t> flags(d->Dslots, 0);
    int dmax = 0;
    for (int k = 0; k < d->Dslots; ++k) {
        const int stq = d->slot_stored[k];
        const double f = stq < 0 ? -1.0 : frac[stq] / rows_per_slot;
        if (slot_fraction) slot_fraction[k] = float(f);
        if (stq >= 0 && f <= double(max_fraction)) {
            flags[k] = 1;
            dmax = std::max(dmax, maxc[stq]);
        }
    }
    const std::vector<uint8_t> old_flags = d->slot_delta;
    d->slot_delta = flags;
    splice_status s2 = replan(d);
    if (s2 == SPLICE_OK) s2 = upload_tables(d, stream);
    if (s2 != SPLICE_OK) {
        d->slot_delta = old_flags;
        replan(d);
        return s2;
    }
    d->delta = b;
    d->delta_max = dmax;
    d->delta_on = std::any_of(flags.begin(), flags.end(), [](uint8_t f) { return f != 0; });
    d->map_ptr[4] = d->map_ptr[5] = nullptr;
    return SPLICE_OK;
}

splice_status splice_delta_clear(splice_desc* d, void* stream) {
    if (!d) return fail(SPLICE_EINVAL, "descriptor is NULL");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    std::fill(d->slot_delta.begin(), d->slot_delta.end(), uint8_t(0));
    splice_status st = replan(d);
    if (st == SPLICE_OK) st = upload_tables(d, stream);
    d->delta_on = false;
    d->delta = nullptr;
    d->delta_max = 0;
    d->map_ptr[4] = d->map_ptr[5] = nullptr;
    return st;
}

splice_status splice_debug_plan_delta(splice_desc* d, const uint8_t* slot_delta) {
    if (!d || !slot_delta) return fail(SPLICE_EINVAL, "NULL descriptor or flags");
    if (d->on_device) return fail(SPLICE_ESTATE, "only host-only descriptors take delta flags without an encoding");
    for (int k = 0; k < d->Dslots; ++k) d->slot_delta[k] = (slot_delta[k] && d->slot_stored[k] >= 0) ? 1 : 0;
    return replan(d);
}

splice_status splice_debug_plan_rows(const splice_desc* d, int layer, int step, int32_t* out, int capacity,
                                     int* num_rows) {
    if (!d || !num_rows) return fail(SPLICE_EINVAL, "NULL descriptor or count");
    if (layer < 0 || layer >= d->shape.num_layers) return fail(SPLICE_EINVAL, "layer %d out of range", layer);
    if (step < 0 || step > d->T) return fail(SPLICE_EINVAL, "step %d not in [0, %d]", step, d->T);
    const Plan& pl = d->plan;
    const int tab = pl.table_of(layer, step);
    const int t0 = pl.table_tile_off[tab], t1 = pl.table_tile_off[tab + 1];
    int n = 0;
    for (int t = t0; t < t1; ++t) n += pl.tiles[4 * size_t(t) + 2];
    *num_rows = n;
    if (!out) return SPLICE_OK;
    if (capacity < n) return fail(SPLICE_EINVAL, "capacity %d < %d rows", capacity, n);
    int r = 0;
    for (int t = t0; t < t1; ++t) {
        const int grp = pl.tiles[4 * size_t(t)], first = pl.tiles[4 * size_t(t) + 1], cnt = pl.tiles[4 * size_t(t) + 2];
        for (int i = 0; i < cnt; ++i, ++r) {
            out[4 * size_t(r) + 0] = t - t0;
            out[4 * size_t(r) + 1] = pl.group_src[grp];
            out[4 * size_t(r) + 2] = pl.group_seqs[first + i];
            out[4 * size_t(r) + 3] = pl.group_mask[first + i];
        }
    }
    return SPLICE_OK;
}

splice_status splice_debug_source_map(splice_desc* d, int layer, int step, uint8_t* host_out) {
    if (!d || !host_out) return fail(SPLICE_EINVAL, "NULL descriptor or output");
    if (layer < 0 || layer >= d->shape.num_layers) return fail(SPLICE_EINVAL, "layer %d out of range", layer);
    if (step < 0 || step > d->T) return fail(SPLICE_EINVAL, "step %d not in [0, %d]", step, d->T);
    const int tab = d->plan.table_of(layer, step);
    if (!d->on_device) {
        std::memcpy(host_out, d->plan.src.data() + size_t(tab) * d->B, d->B);
        return SPLICE_OK;
    }
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaMemcpy(host_out, d->d_src + size_t(tab) * d->B, d->B, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy of the source map");
    return SPLICE_OK;
}

splice_status splice_debug_pass_order(splice_desc* d, int order) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (order < 0 || order > 2) return fail(SPLICE_EINVAL, "pass order %d not in [0, 2]", order);
    d->pass_order = order;
    return SPLICE_OK;
}

splice_status splice_plan_stats(const splice_desc* d, int layer, int step, int* num_groups, int* num_tiles,
                                int* prompt_visible, int* suffix_visible) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (layer < 0 || layer >= d->shape.num_layers) return fail(SPLICE_EINVAL, "layer %d out of range", layer);
    if (step < 0 || step > d->T) return fail(SPLICE_EINVAL, "step %d not in [0, %d]", step, d->T);
    const int tab = d->plan.table_of(layer, step);
    const splice::Visible v = splice::visible_keys(d->shape, d->Tp, layer, step);
    if (num_groups) *num_groups = d->plan.table_group_off[tab + 1] - d->plan.table_group_off[tab];
    if (num_tiles) *num_tiles = d->plan.table_tile_off[tab + 1] - d->plan.table_tile_off[tab];
    if (prompt_visible) *prompt_visible = v.p_hi - v.p_lo;
    if (suffix_visible) *suffix_visible = v.s_hi - v.s_lo;
    return SPLICE_OK;
}

splice_status splice_check_device_error(splice_desc* d) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
    unsigned flag = 0;
    e = cudaMemcpy(&flag, d->d_err, sizeof flag, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemcpy of the error flag");
    if (flag) {
        const unsigned zero = 0;
        cudaMemcpy(d->d_err, &zero, sizeof zero, cudaMemcpyHostToDevice);
        return fail(SPLICE_EDEVICE, "kernel recorded error code 0x%x", flag);
    }
    return SPLICE_OK;
}

splice_status splice_debug_wait_timeout(splice_desc* d, unsigned limit_us, void* stream) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    if (limit_us == 0 || limit_us > 1000000u) return fail(SPLICE_EINVAL, "limit_us %u not in [1, 1000000]", limit_us);
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    cudaError_t e = cudaError_t(splice::launch_wait_timeout(d->d_err, 1000ull * limit_us, stream));
    if (e != cudaSuccess) return cuda_fail(e, "wait-timeout launch");
    return SPLICE_OK;
}

splice_status splice_debug_late_copy(void* dst, const void* src, size_t bytes, unsigned delay_us, void* stream) {
    if (!dst || !src || !aligned16(dst) || !aligned16(src) || bytes % 16 != 0)
        return fail(SPLICE_EINVAL, "splice_debug_late_copy: NULL or misaligned buffer, or bytes not a multiple of 16");
    if (delay_us > 1000000u) return fail(SPLICE_EINVAL, "delay_us %u above 1000000", delay_us);
    cudaError_t e = cudaError_t(splice::launch_late_copy(dst, src, bytes, 1000ull * delay_us, stream));
    if (e != cudaSuccess) return cuda_fail(e, "late-copy launch");
    return SPLICE_OK;
}

long long splice_kernel_launches(const splice_desc* d) { return d ? d->launches : -1; }

splice_status splice_profile_enable(splice_desc* d, int enable) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    d->profiling = enable != 0;
    return SPLICE_OK;
}

splice_status splice_profile_read(splice_desc* d, long long* launches, double* total_ms) {
    if (!d) return fail(SPLICE_EINVAL, "NULL descriptor");
    if (!d->on_device) return fail(SPLICE_ESTATE, "host-only descriptor");
    DeviceGuard g(d->device);
    if (g.err != cudaSuccess) return cuda_fail(g.err, "cudaSetDevice");
    for (int k = 0; k < SPLICE_KERNEL_KINDS; ++k) {
        double ms = 0.0;
        for (size_t i = 0; i < d->events_used[k]; ++i) {
            cudaError_t e = cudaEventSynchronize(d->events[k][i].second);
            if (e != cudaSuccess) return cuda_fail(e, "cudaEventSynchronize");
            float f = 0.f;
            e = cudaEventElapsedTime(&f, d->events[k][i].first, d->events[k][i].second);
            if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
            ms += f;
        }
        if (launches) launches[k] = (long long)d->events_used[k];
        if (total_ms) total_ms[k] = ms;
        d->events_used[k] = 0;
    }
    return SPLICE_OK;
}

const char* splice_kernel_kind_name(int kind) {
    static const char* names[SPLICE_KERNEL_KINDS] = {"append", "prompt_span_pass", "generated_span_pass", "merge"};
    return kind >= 0 && kind < SPLICE_KERNEL_KINDS ? names[kind] : "unknown";
}

}  // extern "C"
