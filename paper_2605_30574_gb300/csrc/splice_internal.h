// Internal declarations of the spliced decode-attention library (not part of
// the C ABI).  Host planner types, kernel parameter blocks and launchers.
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include <vector_types.h>

#include "../../include/splice.h"

namespace splice {

// Largest number of key splits per row for the prompt span and for the
// generated span; the workspace holds kMaxSplits partial states per row.
constexpr int kMaxPrefixSplits = 8;
constexpr int kMaxSuffixSplits = 8;
constexpr int kMaxSplits = kMaxPrefixSplits + kMaxSuffixSplits;
// Rows of one tensor-core prefix tile (tcgen05 M).
constexpr int kTileRows = 128;
// Prompt-span splits: a span's first split holds kPrefixFirstSplitKeys keys,
// every later one kPrefixSplitKeys (the last possibly fewer).
constexpr int kPrefixFirstSplitKeys = 2048;
constexpr int kPrefixSplitKeys = 1024;
// The call's prompt-span pass goes first when it holds fewer than this many
// keys (summed over its items) per SM.
constexpr int kPrefixFirstKeysPerSm = 3072;
// It also goes first when its keys exceed kPrefixFirstGenRatio x the
// generated-span pass's (keys x row chunks).
constexpr int kPrefixFirstGenRatio = 2;
// Group source flag: the group reads the delta-encoded rows of a donor slot
// (group_src = kGroupDelta | (SPLICE_SRC_DONOR0 + slot)).
constexpr int32_t kGroupDelta = SPLICE_GROUP_DELTA;

// Host-side resolution of the splice rule (§3, Algorithm 1) into tables.
//
// Epoch e covers steps [epoch_bounds[e], epoch_bounds[e+1]) where the bounds
// are 0 and every distinct W <= max_steps; layer class c covers layers
// [class_bounds[c], class_bounds[c+1]) with bounds 0 and every distinct
// L < N.  Within one (epoch, class) pair every sequence reads one source.
//
// Delta mode (a slot flagged in slot_delta): a reader of that slot's donor
// joins the (prompt, CLEAN) group with row mask = its stored slot index + 1
// (the prompt-span pass drops the slot's encoded positions from the clean
// span for its rows) and also forms a (prompt, kGroupDelta | source) group
// over the slot's encoded rows.  Groups of stored spans come first in every
// table, delta groups after them.
struct Plan {
    std::vector<int> epoch_bounds;
    std::vector<int> class_bounds;
    int num_tables = 0;                  // epochs * classes
    std::vector<uint8_t> src;            // [num_tables][B] source codes
    // (prompt, source) groups of the sequences that read a stored span.
    std::vector<int32_t> table_group_off;   // [num_tables + 1]
    std::vector<int32_t> group_prompt;      // [groups]
    std::vector<int32_t> group_src;         // [groups] source code (CLEAN or DONOR0 + slot)
    std::vector<int32_t> group_first;       // [groups] offset into group_seqs
    std::vector<int32_t> group_count;       // [groups]
    std::vector<int32_t> group_seqs;        // concatenated sequence indices
    std::vector<int32_t> group_mask;        // parallel to group_seqs: 0, or stored slot + 1 (delta rows)
    // Row tiles of at most kTileRows rows (seqs_per_tile sequences x G heads).
    std::vector<int32_t> table_tile_off;    // [num_tables + 1]
    std::vector<int32_t> tiles;             // [tiles][4]: group, first, count, (span base << 2) | store kind
    std::vector<int32_t> table_span_tiles;  // [num_tables] tiles of stored-span groups (the rest read delta rows)
    int seqs_per_tile = 0;

    int table_of(int layer, int step) const;
};

// slot_delta: [num_donor_slots] nonzero = the slot is read in delta mode
// (NULL = no slot).
std::string build_plan(const splice_model_shape& shape, int num_prompts, int prompt_len,
                       int num_donor_slots, const splice_donor_kind* kinds, int num_seqs,
                       const splice_seq* seqs, int max_steps, const uint8_t* slot_delta, Plan& plan);

// Visible key ranges of the step-t query at layer l: prompt positions
// [p_lo, prompt_len) and generated entries [s_lo, step).
struct Visible {
    int p_lo, p_hi, s_lo, s_hi;
};
Visible visible_keys(const splice_model_shape& shape, int prompt_len, int layer, int step);

// Parameter block of the attention kernels.
struct AttnParams {
    const uint16_t* q;
    const uint16_t* kc;
    const uint16_t* vc;
    const uint16_t* kd;
    const uint16_t* vd;
    const uint16_t* ks;
    const uint16_t* vs;
    // fused append (fuse_append != 0): this step's entries [B][Hkv][D], written
    // by the generated-span pass to entry step - 1 of ks_w / vs_w (the same
    // store as ks / vs) and read from registers instead of from the store
    const uint16_t* kn;
    const uint16_t* vn;
    uint16_t* ks_w;
    uint16_t* vs_w;
    float* out;
    float2* ws_ml;          // [kMaxSplits][B * Hq] (m in log2 units, l)
    float* ws_o;            // [kMaxSplits][B * Hq][D]
    const uint8_t* src;     // [B] source code of every sequence at this (layer, step)
    const int32_t* seq_prompt;
    const int32_t* slot_stored;   // [num_slots] stored-donor index or -1
    const int32_t* seq_slot;      // [B]
    const int32_t* tiles;         // tcgen05 prefix: [n_tiles][4] for this table
    const int32_t* group_prompt;
    const int32_t* group_src;
    const int32_t* group_seqs;
    // delta mode (delta_on != 0)
    const int32_t* group_mask;    // parallel to group_seqs
    const uint32_t* dmask;        // [P][Dst][N][Hkv][delta_w32] encoded-position bits
    const int32_t* dcount;        // [P][Dst][N][Hkv] encoded rows per span
    const int32_t* slot_delta;    // [num_slots] 1 = the slot is read in delta mode
    unsigned* err;
    unsigned* sched;              // [8]: [0], [1] prompt-span work counter and finished-CTA count (zero
                                  // between launches); [2] generated-span claim counter and [4]
                                  // prompt-span pass complete (gs_merge), both cleared by the prompt-span
                                  // pass ahead
    int B, N, Hq, Hkv, D, G, Tp, T, Dst;
    int layer, step;
    int p_lo, p_hi, s_lo, s_hi;
    int nsp, nss;                 // splits of the prompt span / generated span
    int nsd;                      // splits of the delta rows (delta mode)
    int delta_on, delta_w32;
    int fuse_append;              // the generated-span pass also appends entry step - 1 (see kn, vn)
    int gs_after_prefix;          // the generated-span pass runs behind the prompt-span pass of the call
    int prefix_after_gs;          // the prompt-span pass runs behind the generated-span pass of the call
    int gs_merge;                 // the generated-span pass merges rows itself (see launch_generated_span)
    int p_chunk, s_chunk;         // keys per split
    int n_tiles;
    int n_span_tiles;             // tiles [0, n_span_tiles) read stored spans, the rest delta rows
    float scale_log2;             // sm_scale * log2(e)
};

// Records the one-line reason splice_last_error() reports on this thread.
void set_last_error(const char* msg);

// The device a (device) descriptor was created on and launches on; -1 for a
// host-only descriptor or NULL.
int desc_device(const splice_desc* d);

// Launchers (return the cudaError_t of the launch as int).
int launch_append(const uint16_t* kn, const uint16_t* vn, uint16_t* ks, uint16_t* vs, int B,
                  int N, int Hkv, int D, int T, int layer, int step, void* stream);
// overlap_previous: launched as a programmatic dependent of the preceding
// work on the stream.  With p.gs_after_prefix = 0 the kernel is the call's
// first and waits for that work before reading or writing anything, then
// lets its dependents launch.  With 1 it directly follows the prompt-span
// pass of the same call, which has already waited; it reads what that pass
// writes only with p.gs_merge, after it has seen that pass's completion
// flag (sched[4]) and fenced, waits for it only before it exits, and lets
// its own dependents launch only once its work is done.
int launch_generated_span(const AttnParams& p, void* stream, bool overlap_previous);
int generated_span_resident_warps(int d);
// Whether the generated-span pass is built with its merge path for head
// dim d and GQA group G (AttnParams::gs_merge may be set only then).
bool generated_span_can_merge(int d, int G);
// overlap_previous: the launch directly follows the last pass of the same
// call on the stream (programmatic dependent launch; the kernel waits for it,
// and that pass's completion implies the other pass's).
int launch_merge(const AttnParams& p, void* stream, bool overlap_previous);

// A copy of `bytes` (a multiple of 16) from src to dst by a kernel that lets
// its programmatic dependents launch at its start and copies only after
// delay_ns.
int launch_late_copy(void* dst, const void* src, size_t bytes, unsigned long long delay_ns, void* stream);

// One-thread kernel whose mbarrier wait runs out after limit_ns.
int launch_wait_timeout(unsigned* err, unsigned long long limit_ns, void* stream);

// Tensor-core prompt-span pass.  A tensor map is a 128-byte CUtensorMap.
int make_kv_tensor_map(void* out_map, const void* base, long rows, int d, int box_rows);
int prefix_tc_box_rows(int d);
// Key splits of a visible span of p_vis keys: returns their number n (at
// most max_splits) and writes bounds[0 .. n], 0 = bounds[0] < ... <
// bounds[n] = p_vis, every inner bound a multiple of the key block.
int prefix_tc_splits(int d, int p_vis, int max_splits, int* bounds);
// maps: six tensor maps -- clean K, V; donor K, V; delta rows K, V.
// bounds: the span splits (p.nsp + 1 values); delta_keys: keys per split of
// the delta rows.  overlap_previous: a programmatic dependent launch of the
// preceding work on the stream.  With p.prefix_after_gs = 0 the kernel is
// the call's first: it waits for that work before it reads anything, then
// lets its dependents (the generated-span pass) launch onto the SMs its CTAs
// leave.  With 1 it directly follows the generated-span pass of the call,
// which has already waited and lets it start on the SMs that pass's last
// CTAs leave; it reads nothing that pass writes and waits for it before it
// exits.
int launch_prefix_tc(const AttnParams& p, const void* maps, const int* bounds, int delta_keys, void* stream,
                     bool overlap_previous);

// Delta encoding of every stored donor span (one CTA per span): bits of the
// positions whose K or V row differs from the clean span, their count, and
// the donor rows at those positions compacted to the front of the span's
// rows in the delta store (the remaining rows zeroed).
int launch_delta_build(const uint16_t* kc, const uint16_t* vc, const uint16_t* kd, const uint16_t* vd,
                       uint32_t* mask, int32_t* count, uint16_t* xk, uint16_t* xv, int P, int Dst, int N,
                       int Hkv, int Tp, int D, int w32, void* stream);

}  // namespace splice
