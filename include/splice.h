/*
 * splice.h -- C ABI of the GB300-native spliced decode-attention library.
 *
 * The method (arxiv 2605.30574, §3 "Splice intervention", Table 1,
 * Algorithm 1): a chat model with N layers is prefilled on a prompt of
 * length T_p, giving a prompt-span cache K, V at every layer.  During decode
 * step t the model attends over the prompt span concatenated with the t
 * generated-span entries.  One intervention is parameterised by a layer
 * cutoff L (patched layers {l : l >= L}), a splice onset W (steps t < W use
 * the clean span; at t = W the span of every patched layer is replaced in
 * place and stays replaced), and a donor cache (Table 1: ZERO, BLANK,
 * SAME_ALGO, DIFF_ALGO, DIFF_FAMILY).  Generated-span entries are never
 * modified.
 *
 * This library runs a whole (L, W, donor) sweep as one decode batch: every
 * sequence is one sweep cell on one prompt, and each sequence's prompt span
 * is read *by reference* from a shared clean store or a shared donor store,
 * so no spliced cache is ever materialised.
 *
 * Conventions shared by every call
 *   - Tensors are device pointers to dense row-major arrays in the layouts
 *     stated below; bf16 tensors hold IEEE bfloat16 bit patterns
 *     (splice_bf16).  Every tensor pointer must be 16-byte aligned.
 *   - The caller owns every tensor, the workspace and the stream.  The
 *     library owns only the descriptor and its device tables.
 *   - `stream` is a cudaStream_t passed as void*; NULL is the legacy default
 *     stream.  Launch calls are asynchronous on that stream and never
 *     synchronise (except splice_debug_source_map, splice_delta_build and
 *     splice_check_device_error, which say so).
 *   - Every call returns a status and never aborts; CUDA errors raised
 *     asynchronously by earlier launches surface as SPLICE_ECUDA on a later
 *     call.  splice_last_error() gives a one-line reason for the last
 *     failure on the calling thread.
 *   - A descriptor is not thread-safe: do not use one descriptor from two
 *     host threads at once.  Launches that use one descriptor must not
 *     overlap on the GPU either (issue them on one stream, or order them
 *     with events): its device tables hold the error word and the work
 *     counter that the prompt-span pass hands out work with.
 */
#ifndef SPLICE_H
#define SPLICE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t splice_bf16;

typedef enum {
    SPLICE_OK = 0,
    SPLICE_EINVAL = 1,   /* bad argument: shape, range, NULL or misaligned pointer, short workspace */
    SPLICE_ENOMEM = 2,   /* host or device allocation failed */
    SPLICE_ECUDA = 3,    /* a CUDA runtime call failed, or an earlier launch failed asynchronously */
    SPLICE_ESTATE = 4,   /* the descriptor cannot be used this way (host-only descriptor given to a launch) */
    SPLICE_EDEVICE = 5   /* a kernel recorded an error (a bounded wait ran out) */
} splice_status;

/* Donor kinds, Table 1.  ZERO is the all-zero K, V (not stored); the other
 * four are donor caches stored in the donor store. */
typedef enum {
    SPLICE_DONOR_ZERO = 0,
    SPLICE_DONOR_BLANK = 1,
    SPLICE_DONOR_SAME_ALGO = 2,
    SPLICE_DONOR_DIFF_ALGO = 3,
    SPLICE_DONOR_DIFF_FAMILY = 4
} splice_donor_kind;

/* Model shape (§3: N layers, head dim d).  Grouped-query attention: q head h
 * reads kv head floor(h / G), G = num_q_heads / num_kv_heads. */
typedef struct {
    int num_layers;      /* N >= 1 */
    int num_q_heads;     /* Hq, a multiple of num_kv_heads, Hq / Hkv <= 16 */
    int num_kv_heads;    /* Hkv >= 1 */
    int head_dim;        /* d: 64, 128 or 256 */
    int sliding_window;  /* 0 = none; else key j is visible to the step-t query iff
                            (T_p + t - 1) - j < sliding_window on local layers */
    int global_every;    /* with a window: layer l is global (no window) iff
                            (l + 1) % global_every == 0; 0 = every layer local */
    float sm_scale;      /* logit = sm_scale * q . k */
} splice_model_shape;

/* One sweep cell applied to one prompt (§3): the sequence reads the donor
 * span of `donor_slot` at layers l >= L from decode step t >= W on, and the
 * clean span of `prompt_id` otherwise.  W = 0 means replaced before step 1;
 * L >= num_layers or W > max_steps means never replaced. */
typedef struct {
    int prompt_id;       /* 0 <= prompt_id < num_prompts */
    int donor_slot;      /* 0 <= donor_slot < num_donor_slots */
    int L;               /* >= 0 */
    int W;               /* >= 0 */
} splice_seq;

typedef struct splice_desc splice_desc;

/* Source codes written by splice_debug_source_map. */
#define SPLICE_SRC_CLEAN 0u
#define SPLICE_SRC_ZERO 1u
#define SPLICE_SRC_DONOR0 2u     /* donor slot k -> SPLICE_SRC_DONOR0 + k */

/*
 * splice_desc_create -- build the per-sequence splice descriptor of one
 * decode batch (§3; Algorithm 1's Require line: model, prompt span T_p,
 * donor, L, W, max new tokens).
 *
 * The rule "layer l at step t reads the donor iff l >= L and t >= W" is
 * resolved on the host into tables keyed by (epoch, layer class): epochs are
 * the step ranges between distinct W values, layer classes the layer ranges
 * between distinct L values, so every (layer, step) maps to one table in
 * O(log #W).  Each table holds the source of every sequence and the groups
 * of sequences that read the same (prompt, source) span.  The tables are
 * copied to the device on `stream` (asynchronously; the host copies are
 * kept until the copy is complete).
 *
 * Store layouts the later calls assume (bf16):
 *   clean store   [num_prompts][N][Hkv][prompt_len][d]
 *   donor store   [num_prompts][D_stored][N][Hkv][prompt_len][d], where the
 *                 stored slots are the non-ZERO slots in slot order
 *                 (D_stored = splice_num_stored_donor_slots()).
 *
 * num_seqs >= 1, num_prompts >= 1, prompt_len >= 1, 1 <= num_donor_slots
 * <= 250, max_steps >= 1.  The clean and donor stores must each hold fewer
 * than 2^31 rows of d elements.  On success *out owns the descriptor; on
 * failure *out is NULL.
 */
splice_status splice_desc_create(const splice_model_shape* shape, int num_prompts, int prompt_len,
                                  int num_donor_slots, const splice_donor_kind* slot_kinds,
                                  int num_seqs, const splice_seq* seqs, int max_steps,
                                  void* stream, splice_desc** out);

/* Same as splice_desc_create but builds the host tables only (no CUDA call).
 * Such a descriptor answers splice_debug_source_map and the size queries;
 * launch calls on it return SPLICE_ESTATE.  For planning and CPU tests. */
splice_status splice_desc_create_host(const splice_model_shape* shape, int num_prompts,
                                       int prompt_len, int num_donor_slots,
                                       const splice_donor_kind* slot_kinds, int num_seqs,
                                       const splice_seq* seqs, int max_steps, splice_desc** out);

/* Free the descriptor and its device tables.  The caller must make sure no
 * launch that uses it is still in flight.  NULL is accepted. */
splice_status splice_desc_destroy(splice_desc* desc);

/* Bytes of workspace spliced_decode_attn needs for this descriptor (0 for
 * NULL).  The workspace holds per-row partial softmax states; its contents
 * need no initialisation and are meaningless between calls. */
size_t splice_workspace_bytes(const splice_desc* desc);

/* Number of stored (non-ZERO) donor slots, D_stored (-1 for NULL). */
int splice_num_stored_donor_slots(const splice_desc* desc);

/*
 * suffix_kv_append -- append decode step `step`'s generated K, V of every
 * sequence to the generated-span store at slot step - 1 (Algorithm 1's
 * forward pass appends the generated KV to the cache; §3: generated-span
 * entries are never modified afterwards).
 *
 *   k_new, v_new        [num_seqs][Hkv][d] bf16, this step's entries of `layer`
 *   k_suffix, v_suffix  [num_seqs][N][Hkv][max_steps][d] bf16 generated-span store
 *
 * 0 <= layer < N, 1 <= step <= max_steps.  Bit-exact copy.
 */
splice_status suffix_kv_append(splice_desc* desc, int layer, int step, const splice_bf16* k_new,
                               const splice_bf16* v_new, splice_bf16* k_suffix,
                               splice_bf16* v_suffix, void* stream);

/*
 * spliced_decode_attn -- decode attention of every sequence at one layer and
 * one step, over its prompt span (read by reference from the clean store,
 * the donor store, or the ZERO closed form: logit 0 and value 0 at every
 * visible prompt position, Table 1) concatenated with its own first `step`
 * generated entries (§3).
 *
 *   q                   [num_seqs][Hq][d] bf16, queries of this layer and step
 *   k_clean, v_clean    clean store (layout above)
 *   k_donor, v_donor    donor store (layout above); may be NULL when no slot is stored
 *   k_suffix, v_suffix  generated-span store, slots 0 .. step-1 valid
 *   out                 [num_seqs][Hq][d] fp32, softmax(sm_scale q K^T) V per q head
 *   workspace           device scratch of at least splice_workspace_bytes(desc) bytes,
 *                       16-byte aligned (the library places its arrays on 256-byte
 *                       boundaries inside it; the size includes that slack)
 *
 * 0 <= layer < N, 0 <= step <= max_steps (step 0 = empty generated span, a
 * degenerate case for tests; a row with no visible key outputs 0).
 * bf16 inputs, fp32 accumulation and output.
 */
splice_status spliced_decode_attn(splice_desc* desc, int layer, int step, const splice_bf16* q,
                                  const splice_bf16* k_clean, const splice_bf16* v_clean,
                                  const splice_bf16* k_donor, const splice_bf16* v_donor,
                                  const splice_bf16* k_suffix, const splice_bf16* v_suffix,
                                  float* out, void* workspace, size_t workspace_bytes,
                                  void* stream);

/*
 * spliced_decode_step -- one layer of one decode step: suffix_kv_append of
 * (k_new, v_new) at entry step - 1 followed by spliced_decode_attn (Algorithm
 * 1's loop body: the forward pass appends the step's generated K/V, then
 * attends over the prompt span and the step's generated entries, §3), in
 * fewer launches.  The generated-span pass writes the new entries into the
 * store itself and reads them from its registers, so no separate append
 * kernel runs.
 *
 *   k_new, v_new        [num_seqs][Hkv][d] bf16, this step's entries of `layer`
 *   k_suffix, v_suffix  generated-span store; slots 0 .. step-2 valid on entry,
 *                       slot step-1 written by this call
 *   other arguments     as spliced_decode_attn
 *
 * 1 <= step <= max_steps.  Outputs and the store afterwards are bit-identical
 * to suffix_kv_append + spliced_decode_attn on the same inputs.
 */
splice_status spliced_decode_step(splice_desc* desc, int layer, int step, const splice_bf16* q,
                                  const splice_bf16* k_new, const splice_bf16* v_new,
                                  const splice_bf16* k_clean, const splice_bf16* v_clean,
                                  const splice_bf16* k_donor, const splice_bf16* v_donor,
                                  splice_bf16* k_suffix, splice_bf16* v_suffix, float* out,
                                  void* workspace, size_t workspace_bytes, void* stream);

/*
 * spliced_decode_attn_static -- spliced_decode_attn for callers that cannot
 * allocate device memory.  The paper has no counterpart; this is a
 * deployment convenience.
 *
 * Some callers may not call cudaMalloc themselves: for example a plugin
 * inside a host runtime that owns every device allocation through its own
 * memory pool and hands the plugin only the tensors of the call, or a
 * latency-critical decode loop in which an allocation (which can synchronise
 * the device) is not acceptable.  Such a caller passes the same inputs and
 * output as to spliced_decode_attn but no workspace: the partial softmax
 * states live in a file-scope device array of SPLICE_STATIC_SCRATCH_BYTES
 * (64 MiB) inside the library, which every GPU that loads the library holds
 * until the process exits.  This call allocates nothing.
 *
 *   - The scratch used is the array of the descriptor's device (the device
 *     it was created on, where its kernels run); q on another device is
 *     rejected with SPLICE_EINVAL.
 *   - The first call on a device looks up that array's device address (with
 *     that device made current), and looks it up again after the device's
 *     context changed (a cudaDeviceReset); make that first call before any
 *     stream capture.
 *   - A descriptor whose splice_workspace_bytes() exceeds
 *     SPLICE_STATIC_SCRATCH_BYTES is rejected with SPLICE_EINVAL (reduce the
 *     batch, or use spliced_decode_attn with a workspace).
 *     splice_static_scratch_bytes() returns that limit as built.
 *   - Every call on a device shares the one array, and it keeps the last
 *     call's contents; nothing in it needs to start at zero.  Calls that
 *     overlap on the GPU (other streams, other host threads, other
 *     descriptors) race on it: serialise them.
 *
 * Arguments, layouts and errors are otherwise those of spliced_decode_attn.
 */
#define SPLICE_STATIC_SCRATCH_BYTES (64u << 20)
size_t splice_static_scratch_bytes(void);
splice_status spliced_decode_attn_static(splice_desc* desc, int layer, int step, const splice_bf16* q,
                                         const splice_bf16* k_clean, const splice_bf16* v_clean,
                                         const splice_bf16* k_donor, const splice_bf16* v_donor,
                                         const splice_bf16* k_suffix, const splice_bf16* v_suffix,
                                         float* out, void* stream);

/*
 * Delta-donor encoding.  The paper has no counterpart; it changes how a donor
 * span is read, not what is computed.
 *
 * Table 1's donors are aligned position by position with the clean prompt
 * (§3 trims donor and target prompts to the same length), and a donor may
 * share many positions with it bit for bit (the synthetic donor-noise
 * ladder's SAME_ALGO / DIFF_ALGO donors keep 90% / 50% of their content
 * positions).  Reading such a donor span re-reads bytes that the clean
 * span's readers read anyway.  The delta encoding of a stored donor span
 * against the clean span of the same prompt, layer and kv head is the set of
 * positions whose K row or V row differs bit for bit, as a bitmask, and the
 * donor's rows at those positions in increasing position order.  It is
 * lossless, and attention over the donor span equals the log-sum-exp merge
 * of attention over the clean span without those positions and attention
 * over the encoded rows.  In delta mode the readers of an encoded slot are
 * stacked into the clean span's tiles (their encoded positions dropped row
 * by row) and read the encoded rows as tiles of their own.
 *
 * splice_delta_bytes -- bytes of the delta buffer of this descriptor (0 for
 * NULL or when no slot is stored).  Layout, each part starting on a 256-byte
 * boundary in this order (W32 = 4 * ceil(prompt_len / 128) words per span):
 *   mask    [num_prompts][D_stored][N][Hkv][W32] uint32: bit j % 32 of word
 *           j / 32 set iff position j is encoded
 *   count   [num_prompts][D_stored][N][Hkv] int32: encoded positions
 *   rows_k  [num_prompts][D_stored][N][Hkv][prompt_len][d] bf16: rows
 *           0 .. count-1 hold the encoded donor rows, the rest zeros
 *   rows_v  same, for V
 *
 * splice_delta_build -- encode every stored donor span on `stream`, read the
 * counts back (this synchronises the stream), and put the descriptor in
 * delta mode for every stored slot whose encoded fraction (encoded positions
 * over all positions of the slot's spans) is at most max_fraction; other
 * slots keep reading the donor store.  slot_fraction (may be NULL) receives
 * num_donor_slots fractions, -1 for ZERO slots.
 *   k_clean, v_clean, k_donor, v_donor  the stores later calls will read
 *   delta         caller-owned device buffer of splice_delta_bytes(desc) bytes
 *   max_fraction  in [0, 1]
 * The caller keeps `delta` and the stores' contents unchanged while the
 * descriptor is in delta mode (encode again after changing a store) and
 * passes the same stores to spliced_decode_attn.  The descriptor's device
 * tables are rebuilt: no launch that uses the descriptor may be in flight.
 * Rejected with SPLICE_EINVAL: a descriptor with a sliding window (the
 * encoded rows carry no positions), one with no stored slot, or a prompt_len
 * above 204800.  Outputs of delta mode meet the same tolerance against exact
 * attention as the default mode but are not bit-identical to it.
 *
 * splice_delta_clear -- leave delta mode (device tables rebuilt on `stream`;
 * no launch that uses the descriptor may be in flight).
 */
size_t splice_delta_bytes(const splice_desc* desc);
splice_status splice_delta_build(splice_desc* desc, const splice_bf16* k_clean, const splice_bf16* v_clean,
                                 const splice_bf16* k_donor, const splice_bf16* v_donor, void* delta,
                                 size_t delta_bytes, float max_fraction, float* slot_fraction, void* stream);
splice_status splice_delta_clear(splice_desc* desc, void* stream);

/*
 * Planner views for tests (host tables only, no CUDA call).
 *
 * splice_debug_plan_delta -- host-only descriptors: re-plan as if the slots
 * flagged in slot_delta (num_donor_slots bytes; ZERO slots ignored) were in
 * delta mode.
 *
 * splice_debug_plan_rows -- the rows of the prompt-span tiles at (layer,
 * step), in tile order: out[4 i ..] = (tile, group source, sequence, row
 * mask), where the group source is SPLICE_SRC_CLEAN, SPLICE_SRC_DONOR0 +
 * slot, or SPLICE_GROUP_DELTA | (SPLICE_SRC_DONOR0 + slot) for the encoded
 * rows of a slot, and the row mask is 0 or, for a delta-mode reader in a
 * clean tile, its stored slot index + 1.  *num_rows receives the count;
 * with out == NULL only the count is returned, else capacity (in rows) must
 * cover it.
 */
#define SPLICE_GROUP_DELTA 0x100
splice_status splice_debug_plan_delta(splice_desc* desc, const uint8_t* slot_delta);
splice_status splice_debug_plan_rows(const splice_desc* desc, int layer, int step, int32_t* out, int capacity,
                                     int* num_rows);

/*
 * splice_debug_source_map -- the prompt-span source every sequence reads at
 * (layer, step): host_out[s] = SPLICE_SRC_CLEAN, SPLICE_SRC_ZERO or
 * SPLICE_SRC_DONOR0 + slot.  For a device descriptor the map is read back
 * from the device tables (this synchronises the device); for a host-only
 * descriptor it comes from the host tables.  host_out has num_seqs bytes.
 */
splice_status splice_debug_source_map(splice_desc* desc, int layer, int step, uint8_t* host_out);

/*
 * splice_plan_stats -- shape of the work at (layer, step), from the host
 * tables: number of (prompt, source) groups that read a stored span, number
 * of 128-row prefix tiles, and the visible prompt positions and generated
 * entries per sequence.  Any output pointer may be NULL.
 */
splice_status splice_plan_stats(const splice_desc* desc, int layer, int step, int* num_groups,
                                int* num_tiles, int* prompt_visible, int* suffix_visible);

/*
 * splice_debug_pass_order -- order of the two attention passes in later
 * calls on the descriptor: 0 (the default) chosen per call from the plan --
 * the prompt-span pass first when it holds fewer than 3072 keys per SM
 * (summed over its items) or more than twice the generated-span pass's
 * keys, else the generated-span pass first; 1 the prompt-span pass first;
 * 2 the generated-span pass first.  Outputs and stores are bit-identical in
 * every order (the passes write disjoint partial states that are combined
 * in a fixed order, by the merge kernel or -- with the prompt-span pass
 * first and one split of each span -- by the generated-span pass once the
 * prompt-span pass has completed); only the overlap of the two passes
 * changes.
 * SPLICE_EINVAL for another value.  No device work.
 */
splice_status splice_debug_pass_order(splice_desc* desc, int order);

/* Synchronise the device and report kernel-side errors recorded since the
 * descriptor was created (SPLICE_EDEVICE), clearing the record. */
splice_status splice_check_device_error(splice_desc* desc);

/*
 * Measurement support.  The library counts the kernels it launches and can
 * bracket each launch with CUDA events recorded on the launch's stream.
 * Kernel kinds: 0 generated-span append, 1 prompt-span pass, 2 generated-
 * span pass, 3 merge (splice_kernel_kind_name gives the names).
 *
 * splice_kernel_launches: kernels launched through this descriptor so far.
 * splice_profile_enable: turn per-launch event timing on (1) or off (0).
 * splice_profile_read: synchronise on the recorded events and return, per
 *   kind (arrays of SPLICE_KERNEL_KINDS), the number of timed launches and
 *   their summed duration in milliseconds since the previous read; then
 *   reset.  Either array may be NULL.
 */
#define SPLICE_KERNEL_KINDS 4
long long splice_kernel_launches(const splice_desc* desc);
splice_status splice_profile_enable(splice_desc* desc, int enable);
splice_status splice_profile_read(splice_desc* desc, long long* launches, double* total_ms);
const char* splice_kernel_kind_name(int kind);

/* Test of the failure path: launches one thread whose mbarrier wait can never
 * complete and gives up after limit_us microseconds (1 .. 1000000), recording
 * an error bit in the descriptor's error word exactly as a streaming kernel's
 * bounded wait would; splice_check_device_error then returns SPLICE_EDEVICE.
 * Nothing faults or hangs. */
splice_status splice_debug_wait_timeout(splice_desc* desc, unsigned limit_us, void* stream);

/* Test of launch ordering: copies `bytes` (a multiple of 16; both pointers
 * 16-byte aligned) from src to dst on `stream` with a kernel that lets its
 * programmatic dependents launch as soon as it starts but copies only after
 * delay_us microseconds (0 .. 1000000) of wall time.  A library call queued
 * right behind it must still read the copied data: every kernel of the
 * library waits for the work before it on the stream before it reads its
 * inputs.  Nothing faults or hangs. */
splice_status splice_debug_late_copy(void* dst, const void* src, size_t bytes, unsigned delay_us, void* stream);

/* Static description of a status code. */
const char* splice_status_str(splice_status status);

/* One-line reason for the last failing call on this thread ("" if none). */
const char* splice_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SPLICE_H */
