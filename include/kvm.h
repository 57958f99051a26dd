/*
 * kvm.h -- C ABI of the true-tail incremental memory maintenance library.
 *
 * The library keeps, for a population of characters, the inference state
 * (A_t, R_t, p_t) of a hybrid gated-delta-rule / GQA-attention model (§4.1):
 *   A_t  live attention KV per attention layer (rotated keys and values,
 *        bf16, plus one int32 position id per live entry, shared by all
 *        attention layers of a character),
 *   R_t  the recurrent state S [H][d_v][d_k] (fp32) of every delta-rule layer,
 *   p_t  the next position id (cursor), which only moves forward (§4.2).
 * A maintenance round removes the KV of superseded records in every attention
 * layer (Eq. 2) and runs the M replacement tokens forward at the true tail
 * (Eq. 3): attention layers append the tail's keys at positions p .. p+M-1
 * and attend causally over the compacted cache plus the tail; delta-rule
 * layers advance S from its preserved value.  Projections, norms and MLPs of
 * the full model are outside this library: callers pass per-layer q/k/v (and
 * the gates alpha, beta) and receive per-layer outputs.
 *
 * Conventions for every entry point:
 *  - Return value: KVM_OK (0) or a KVM_E_* code.  On any error the text of
 *    the failure is available from kvm_last_error() (thread-local), and the
 *    context state is unchanged: all argument and span validation happens on
 *    the host before the first launch.
 *  - "device" pointers are CUDA global-memory addresses on the context's
 *    device; "host" pointers are CPU memory.  bf16 tensors are passed as
 *    void* holding IEEE bfloat16 values.  Every device pointer must be
 *    16-byte aligned.
 *  - stream is a cudaStream_t (NULL = legacy default stream).  Work is
 *    enqueued asynchronously on it; the caller keeps device buffers alive
 *    until that work completes.  A context is used from one host thread and
 *    one stream at a time.
 *  - Characters are packed: per-character token counts are given as
 *    cumulative offsets cu[B+1] (cu[0] = 0), and tensors of tail tokens are
 *    [sum M][heads][dim] with character b's tokens at rows cu[b] .. cu[b+1]-1.
 *  - Kernels never trap.  A bounds violation or an expired bounded wait
 *    detected on the device sets a device error word; kvm_check() reads it.
 */
#ifndef KVM_H
#define KVM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int kvm_status;
enum {
    KVM_OK = 0,
    KVM_E_INVAL = 1,        /* NULL or inconsistent argument, bad layer index */
    KVM_E_SPAN = 2,         /* deletion span unsorted, overlapping, empty or outside the live cache */
    KVM_E_CAPACITY = 3,     /* L' + M exceeds a character's capacity, or sum M exceeds max_tail_tokens */
    KVM_E_CUDA = 4,         /* CUDA runtime / launch failure (text in kvm_last_error) */
    KVM_E_DEVICE = 5,       /* a kernel reported a bounds violation or an expired wait */
    KVM_E_UNSUPPORTED = 6   /* shape outside what the kernels implement */
};

enum { KVM_LAYER_GDN = 0, KVM_LAYER_ATTN = 1 };

typedef struct kvm_ctx kvm_ctx;

/* Model shape.  layer_kind[n_layers] lists the layers in model order.
 * Attention layers: n_q_heads query heads share n_kv_heads KV heads (query
 * head h reads KV head h / (n_q_heads / n_kv_heads)); head_dim D; RoPE on the
 * first rotary_dim dims of each head, pairs (d, d + rotary_dim/2), frequency
 * rope_theta^(-2d/rotary_dim); scores scaled by 1/sqrt(D).
 * Delta-rule layers: n_gdn_heads heads with key dim d_k and value dim d_v.
 * Supported: D in {64, 128, 256}; rotary_dim even, <= D; group size
 * n_q_heads/n_kv_heads a power of two <= 64; d_k in {64, 128}; d_v a
 * multiple of 32, <= 128. */
typedef struct kvm_model_desc {
    int32_t n_layers;
    const int32_t* layer_kind;     /* host [n_layers] */
    int32_t n_q_heads;
    int32_t n_kv_heads;
    int32_t head_dim;
    int32_t rotary_dim;
    double rope_theta;
    int32_t n_gdn_heads;
    int32_t d_k;
    int32_t d_v;
    /* Short convolution of the delta-rule layers (§4.1: R_t holds the
     * recurrent and the convolution states): 0 = none (q, k, v are used as
     * given); 4 = the layer's q, k, v inputs are pre-convolution projections,
     * filtered per channel by a causal depthwise convolution of width 4 over
     * the tail and the last three inputs of earlier rounds (the carried conv
     * state), then SiLU; k is then scaled to unit L2 norm per head.  Weights
     * per layer with kvm_set_conv_weights. */
    int32_t conv_kernel;
} kvm_model_desc;

/* ---------------------------------------------------------------- lifetime */

/* Create a context for n_chars characters on the current CUDA device.
 * capacity: host [n_chars], KV slots per character (every attention layer);
 * max_tail_tokens: upper bound on sum M of any later round (sizes the
 * workspace).  The context allocates all persistent state (KV slabs,
 * positions, S, cursors) and all workspace here, once; later calls allocate
 * nothing.  Initial state: live length 0, cursor 0, S = 0.
 * Errors: KVM_E_INVAL, KVM_E_UNSUPPORTED, KVM_E_CUDA (out of memory). */
kvm_status kvm_create(const kvm_model_desc* model, int32_t n_chars,
                      const int32_t* capacity, int32_t max_tail_tokens,
                      kvm_ctx** out);

/* Free everything the context owns.  Synchronizes the device first. */
kvm_status kvm_destroy(kvm_ctx* ctx);

/* Text of the most recent failure on this host thread ("" if none). */
const char* kvm_last_error(void);

/* ------------------------------------------------------------ state access */

/* Load a character's prefix: live length `live` (<= capacity), cursor p
 * (the next position id; must exceed every position), positions host
 * [live] (strictly increasing, >= 0).  Keys/values are then set per layer
 * with kvm_set_kv.  Synchronous with respect to the host arrays. */
kvm_status kvm_load_prefix(kvm_ctx* ctx, int32_t b, int32_t live, int64_t cursor,
                           const int32_t* positions, void* stream);

/* Copy a character's live KV of attention layer `layer` (model index) in or
 * out.  k, v: device [n_kv_heads][live][head_dim] bf16, keys in stored
 * (already rotated) form. */
kvm_status kvm_set_kv(kvm_ctx* ctx, int32_t layer, int32_t b, const void* k,
                      const void* v, void* stream);
kvm_status kvm_get_kv(kvm_ctx* ctx, int32_t layer, int32_t b, void* k_out,
                      void* v_out, void* stream);

/* Device positions of character b: pos_out device [live] int32. */
kvm_status kvm_get_positions(kvm_ctx* ctx, int32_t b, int32_t* pos_out, void* stream);

/* Recurrent state of delta-rule layer `layer` (model index), all characters:
 * device [n_chars][n_gdn_heads][d_v][d_k] fp32. */
kvm_status kvm_set_state(kvm_ctx* ctx, int32_t layer, const float* S, void* stream);
kvm_status kvm_get_state(kvm_ctx* ctx, int32_t layer, float* S_out, void* stream);

/* Short-convolution weights and state of delta-rule layer `layer` (model
 * index), for contexts created with conv_kernel = 4.  Channels are ordered q
 * [H][d_k], k [H][d_k], v [H][d_v] (C = H (2 d_k + d_v)).
 * kvm_set_conv_weights: w device fp32 [C][4], tap i multiplies the input
 * 3 - i tokens back (tap 3 is the current token); the context keeps a copy.
 * kvm_get_conv_state / kvm_set_conv_state: device bf16 [n_chars][3][C], the
 * last three pre-convolution inputs of each character (oldest first); a new
 * context starts from zeros.  Errors: KVM_E_INVAL (no conv, wrong layer). */
kvm_status kvm_set_conv_weights(kvm_ctx* ctx, int32_t layer, const float* w, void* stream);
kvm_status kvm_get_conv_state(kvm_ctx* ctx, int32_t layer, void* state_out, void* stream);
kvm_status kvm_set_conv_state(kvm_ctx* ctx, int32_t layer, const void* state, void* stream);

/* Host view of character b's live length and cursor (no synchronization). */
kvm_status kvm_get_live(kvm_ctx* ctx, int32_t b, int32_t* live, int64_t* cursor);

/* Map absolute position ranges [pos_begin, pos_end) of character b to
 * live-index spans, checking each against the live entries (§4.2: deletion
 * ranges are verified against live spans).  A range must cover at least one
 * live entry and every live entry whose position lies in it; the ranges
 * must be sorted and disjoint.  When per-token positions or re-rotation have
 * left the live positions out of order, the entries a range covers must form
 * one contiguous run of live indices.  Outputs host [n].  Errors:
 * KVM_E_SPAN. */
kvm_status kvm_spans_from_positions(kvm_ctx* ctx, int32_t b, int32_t n,
                                    const int64_t* pos_begin, const int64_t* pos_end,
                                    int32_t* span_begin, int32_t* span_end);

/* ------------------------------------------------------------ host-only planning
 * These touch no context and no device: they compute on the host what the
 * hot-path calls plan before their first launch, so that a caller can check
 * a round ahead of time and tests can check the planning on a machine
 * without a GPU. */

/* Eq. 2 on the host: validate one round's removal spans against the live
 * lengths live host [n_chars] with exactly the checks of kvm_kv_compact
 * (span_cu, span_begin, span_end as there), and report its effect: new_live
 * host [n_chars] = L'_b = live_b minus the removed count, first_moved host
 * [n_chars] = the first live index at or after which entries move (the first
 * span's begin; L'_b when the character removes nothing).  Either output may
 * be NULL.  Errors: KVM_E_INVAL, KVM_E_SPAN. */
kvm_status kvm_plan_removal(int32_t n_chars, const int32_t* live, const int32_t* span_cu,
                            const int32_t* span_begin, const int32_t* span_end, int32_t* new_live,
                            int32_t* first_moved);

/* kvm_spans_from_positions on a caller's copy of one character's live
 * positions: positions host [live], non-negative, in live order.  Same mapping,
 * checks and errors (KVM_E_INVAL for bad arguments, KVM_E_SPAN for ranges). */
kvm_status kvm_plan_spans_from_positions(int32_t live, const int32_t* positions, int32_t n,
                                         const int64_t* pos_begin, const int64_t* pos_end,
                                         int32_t* span_begin, int32_t* span_end);

/* The work partition kvm_tail_attn_prefill uses for one attention layer
 * (Eq. 3), for live lengths L'_b live host [n_chars] (after removal) and
 * tails tail_cu host [n_chars+1].  Query tiles hold 128 / g tail tokens of
 * one KV head (g = n_q_heads / n_kv_heads) and are numbered (character, KV
 * head, tile); tile t of character b attends to ceil((L'_b + last token of
 * the tile + 1) / 64) 64-key tiles.  The (query tile, key tile) units, in
 * that order, are cut into *n_blocks <= max_blocks contiguous ranges; block
 * c processes units from (block_tile[c], block_key[c]) up to, not including,
 * (block_tile[c+1], block_key[c+1]).  block_tile and block_key: host
 * [max_blocks + 1].  *n_tiles = number of query tiles.  split_first_block
 * host [max_blocks]: for each of the *n_split query tiles that several
 * blocks share, the first block that starts inside it (its partials are
 * merged by the combine kernel).  kvm_tail_attn_prefill uses max_blocks =
 * min(320, the device's SM count).  Errors: KVM_E_INVAL, KVM_E_UNSUPPORTED. */
kvm_status kvm_plan_attention(int32_t n_chars, const int32_t* live, const int32_t* tail_cu,
                              int32_t n_q_heads, int32_t n_kv_heads, int32_t max_blocks,
                              int32_t* n_blocks, int32_t* n_tiles, int32_t* block_tile,
                              int32_t* block_key, int32_t* n_split, int32_t* split_first_block);

/* Partition of a character population over ranks (one GPU per rank):
 * characters are independent, so each rank maintains its own share with no
 * exchange on the data path.  cost host [n_chars] >= 0, e.g. a round's
 * attention work M_b (L'_b + (M_b + 1) / 2), the term the round's time
 * follows.  Longest-processing-time first: characters by decreasing cost
 * (ties by index), each to the rank with the least cost so far (ties: the
 * lowest rank), so the heaviest rank exceeds the mean by less than the
 * largest single cost.  rank_of host [n_chars]; rank_cost host [n_ranks]
 * (may be NULL).  Deterministic: every rank computes the same plan.
 * Errors: KVM_E_INVAL. */
kvm_status kvm_plan_partition(int32_t n_chars, const int64_t* cost, int32_t n_ranks, int32_t* rank_of,
                              int64_t* rank_cost);

/* ------------------------------------------------------------ hot path */

/* Eq. 2: remove the live entries named by the spans from every attention
 * layer of every character, keeping survivors' bytes, positions and order
 * (stored keys are never re-rotated, §4.2).  Survivor at old live index i
 * moves to i - (number of removed indices < i), in place; only entries at or
 * after a character's first removed index move.
 * span_cu: host [n_chars+1] offsets into span_begin/span_end (host), which
 * hold half-open live-index ranges, sorted and disjoint per character.
 * gather_out: optional device int32 [sum L'_b], written new slot -> old slot
 * for every surviving entry, characters packed in order; may be NULL.
 * Errors: KVM_E_INVAL, KVM_E_SPAN (nothing launched, state unchanged). */
kvm_status kvm_kv_compact(kvm_ctx* ctx, const int32_t* span_cu,
                          const int32_t* span_begin, const int32_t* span_end,
                          int32_t* gather_out, void* stream);

/* Eq. 3 for one attention layer (model index `layer`): rotate the tail's
 * queries and keys at positions p_b + i (§4.2, RoPE at the true tail),
 * append rotated keys and values at live slots L'_b + i (L'_b = the current
 * live length, i.e. after kv_compact) and write positions p_b + i, then
 * o_i = sum_j softmax_j(q_i . k_j / sqrt(D)) v_j over every surviving entry
 * and the tail's keys j <= i.
 * tail_cu host [n_chars+1]; q device [sum M][n_q_heads][D] bf16;
 * k_new, v_new device [sum M][n_kv_heads][D] bf16; out device
 * [sum M][n_q_heads][D] bf16.  Does not move live lengths or cursors (see
 * kvm_advance), so every attention layer of a round appends at the same
 * slots.  Errors: KVM_E_INVAL, KVM_E_CAPACITY. */
kvm_status kvm_tail_attn_prefill(kvm_ctx* ctx, int32_t layer, const int32_t* tail_cu,
                                 const void* q, const void* k_new, const void* v_new,
                                 void* out, void* stream);

/* Eq. 3 for one gated-delta-rule layer (model index `layer`): advance each
 * character's carried state S (and, with conv_kernel = 4, first its conv
 * state over the q/k/v inputs, see kvm_model_desc) through its M_b tail tokens,
 *   S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T,
 *   o_t = S_t q_t,
 * computed in chunks of 64 tokens (WY/UT form) starting at the first tail
 * token.  S is updated in place in the context.
 * q, k device [sum M][n_gdn_heads][d_k] bf16 (k expected unit-norm per head
 * but not required); v device [sum M][n_gdn_heads][d_v] bf16; alpha, beta
 * device [sum M][n_gdn_heads] fp32; out device [sum M][n_gdn_heads][d_v]
 * bf16.  Errors: KVM_E_INVAL, KVM_E_CAPACITY. */
kvm_status kvm_gdn_chunk_scan_from_state(kvm_ctx* ctx, int32_t layer, const int32_t* tail_cu,
                                         const void* q, const void* k, const void* v,
                                         const float* alpha, const float* beta,
                                         void* out, void* stream);

/* End of a round: p_b += M_b and L_b = L'_b + M_b for every character
 * (host bookkeeping; the device positions were written by the attention
 * layers).  tail_cu host [n_chars+1]. */
kvm_status kvm_advance(kvm_ctx* ctx, const int32_t* tail_cu);

/* Placement variants of the tail (§5.2: fresh gapped prefill reads the text
 * with gaps between records' position ids; slot-preserving maintenance
 * rotates the replacement's queries and keys at its original slot's ids).
 * As kvm_tail_attn_prefill, but tail token n (packed) is rotated at, and
 * stored with, position id tail_pos[n] (host [sum M], each >= 0; NULL = the
 * true tail p_b + i).  Attention stays causal in processing order: a tail
 * token sees every surviving entry and the tail tokens before it, whatever
 * their ids.  Errors: as kvm_tail_attn_prefill. */
kvm_status kvm_tail_attn_prefill_at(kvm_ctx* ctx, int32_t layer, const int32_t* tail_cu,
                                    const int32_t* tail_pos, const void* q, const void* k_new,
                                    const void* v_new, void* out, void* stream);

/* kvm_advance after kvm_tail_attn_prefill_at: the host position mirror gets
 * tail_pos (host [sum M], NULL = p_b + i) and the cursor moves to
 * max(p_b, largest position + 1), so ids are never reused. */
kvm_status kvm_advance_at(kvm_ctx* ctx, const int32_t* tail_cu, const int32_t* tail_pos);

/* Tail-and-relocate (§5.2, §6.3): after a tail computed at tail positions,
 * turn the stored keys of character b's live entries [live_begin, live_end)
 * in every attention layer from the positions they were rotated at to
 * new_pos (host [live_end - live_begin], each >= 0): each rotary pair of a
 * key is rotated by (new_pos - old position) * omega_d, which for rotations
 * equals rotating the unrotated key at new_pos.  Values, recurrent states
 * and the entries' order are unchanged; the stored positions become new_pos
 * and the cursor moves to max(p_b, largest new position + 1).  The keys are
 * re-rounded to bf16 once.  Errors: KVM_E_INVAL, KVM_E_SPAN (range outside
 * the live entries). */
kvm_status kvm_rerotate_keys(kvm_ctx* ctx, int32_t b, int32_t live_begin, int32_t live_end,
                             const int32_t* new_pos, void* stream);

/* One whole maintenance round (Eq. 2 then Eq. 3 for every layer; §4.1, §4.2):
 * kv_compact, then every layer in model order (tail_attn_prefill or
 * gdn_chunk_scan_from_state), then advance.  Per-layer arrays are indexed by
 * model layer; alpha/beta entries of attention layers are ignored.
 * Ordering: everything the round does is complete when the work enqueued on
 * `stream` up to this call's return has completed.  Internally the
 * compaction may run on a stream of the context beside the recurrent layers
 * that precede the first attention layer (it touches only the attention
 * caches), joined back into `stream` before the first attention layer.
 * io_on_host = 0: q/k/v/alpha/beta/out are device pointers.
 * io_on_host = 1: they are host pointers (pinned memory for asynchronous
 * copies, valid until `stream` has completed the round); the library copies
 * every layer's inputs up into its own device staging buffers on a copy
 * stream at once, each layer waiting only for its own, and each layer's
 * output back while the next layers compute.  Inputs of one layer that lie
 * back to back in host memory (q, k, v, alpha, beta in that order, each
 * padded to 16 bytes) go up in one copy.  Errors: as the per-layer calls,
 * all detected on the host before the first launch. */
typedef struct kvm_round {
    const int32_t* span_cu;        /* host [n_chars+1] */
    const int32_t* span_begin;     /* host */
    const int32_t* span_end;       /* host */
    const int32_t* tail_cu;        /* host [n_chars+1] */
    const void* const* q;          /* [n_layers] */
    const void* const* k;          /* [n_layers] */
    const void* const* v;          /* [n_layers] */
    const float* const* alpha;     /* [n_layers] */
    const float* const* beta;      /* [n_layers] */
    void* const* out;              /* [n_layers] */
    int32_t io_on_host;
    int32_t* gather_out;           /* optional device, see kvm_kv_compact */
    /* Placement variants (§5.2), optional: tail_pos host [sum M] gives each
     * tail token its position id (>= 0) for RoPE and for the stored
     * position; NULL places the tail at the true tail p_b + i.  Attention
     * stays causal in processing order: a tail token sees every surviving
     * entry and the tail tokens before it, whatever their position ids.
     * With tail_pos the cursor moves to max(p_b, largest position + 1). */
    const int32_t* tail_pos;
    /* Maintenance delimiters (§4.2), optional: delim_cu host [n_chars+1]
     * offsets into delim_begin/delim_end (host), half-open tail-index ranges
     * [s, e) within [0, M_b), sorted and disjoint per character.  Those tail
     * tokens are processed like the rest (later tail tokens attend to them,
     * the recurrent states absorb them), then their KV leave every attention
     * layer at the end of the round; their position ids stay consumed.
     * NULL: no delimiters. */
    const int32_t* delim_cu;
    const int32_t* delim_begin;
    const int32_t* delim_end;
} kvm_round;

kvm_status kvm_update_round(kvm_ctx* ctx, const kvm_round* round, void* stream);

/* Allocation-free compaction for callers that cannot call cudaMalloc --
 * for example an engine that owns all device memory through its own fixed
 * arena and forbids other allocations during a session, or a frame loop in
 * which an allocation (which may synchronize the device) would stall the
 * frame.  Such callers cannot create a context, so this call removes the
 * given live-index spans from KV buffers they own, with the same in-place
 * result as kvm_kv_compact.  The paper has no counterpart of this call.
 * K, V: device [n_slabs][slab_rows][head_dim] bf16 (n_slabs = attention
 * layers x KV heads, every slab loses the same rows); positions: device
 * [slab_rows] int32, compacted too, or NULL.  live: rows in use before the
 * call; spans: host [n_spans], sorted, disjoint, inside [0, live).
 * new_live_out (host) receives live minus the removed rows.
 * Scratch: the kernel's bookkeeping lives in a fixed ~260 KB device array
 * inside the library (every GPU that loads the library holds it until the
 * process exits); this call allocates nothing.  Limits: n_slabs <= 512,
 * n_spans <= 1024, head_dim in {64, 128, 256}, and
 * 2 * n_slabs * ceil(moved / (16384 / head_dim)) + ceil(moved / 2048) <= 65536
 * where moved = rows from the first span to the new live end (e.g. 24 slabs
 * of head_dim 256 allow ~87K moved rows); larger requests return
 * KVM_E_CAPACITY.  The first call on each device looks up the array's device
 * address (cudaGetSymbolAddress); make that first call before any stream
 * capture.  Every call shares the one array and clears the part it uses, so
 * calls that may overlap on the GPU (other streams, other host threads on
 * the same device) race: order them.  A device-side wait that expires
 * (which valid arguments never cause) leaves that chunk unmoved and sets a
 * bit in the array's error word; kvm_kv_compact_noalloc_check reads it.
 * Errors: KVM_E_INVAL, KVM_E_SPAN, KVM_E_CAPACITY, KVM_E_UNSUPPORTED,
 * KVM_E_CUDA. */
kvm_status kvm_kv_compact_noalloc(void* K, void* V, int32_t* positions, int32_t n_slabs,
                                  int64_t slab_rows, int32_t head_dim, int32_t live,
                                  int32_t n_spans, const int32_t* span_begin,
                                  const int32_t* span_end, int32_t* new_live_out, void* stream);

/* The failure signal of kvm_kv_compact_noalloc on the current device: waits
 * for `stream`, then reads and clears the error word of the library's
 * static scratch array.  Returns KVM_E_DEVICE if a call since the last check
 * reported a bounds violation or an expired wait (the rows of that call are
 * then undefined), KVM_OK otherwise.  Allocates nothing; the paper has no
 * counterpart of this call.  Errors: KVM_E_DEVICE, KVM_E_CUDA. */
kvm_status kvm_kv_compact_noalloc_check(void* stream);

/* ------------------------------------------------------------ diagnostics */

/* Attention probe (§5.3; Appendix C): how the last n_q query tokens of
 * character b distribute attention over its live KV in attention layer
 * `layer` (model index), reconstructed with a float32 reference softmax.
 * q: device [n_q][n_q_heads][D] bf16, the unrotated queries of the last n_q
 * live entries (the probe tokens, already appended by a round); query i is
 * rotated at the position of live entry L - n_q + i and sees live entries
 * 0 .. L - n_q + i (causal in processing order).  Removed records leave no
 * entries, so the denominator runs over live tokens only (holes excluded).
 * probs_out: device fp32 [L] (L = live length), the probability of each live
 * entry averaged over the n_q queries and all query heads (sums to 1).
 * group_of: optional device int32 [L], a group id in [0, n_groups) per live
 * entry (-1: in no group), e.g. the memory record it belongs to;
 * group_mass_out: device fp32 [n_groups], the summed probability per group.
 * 1 <= n_q <= min(16, L).  Uses the context's workspace; enqueued on
 * `stream`.  Errors: KVM_E_INVAL.  A group id >= n_groups is reported by
 * kvm_check (KVM_E_DEVICE). */
kvm_status kvm_attn_probe(kvm_ctx* ctx, int32_t layer, int32_t b, int32_t n_q, const void* q,
                          float* probs_out, const int32_t* group_of, int32_t n_groups,
                          float* group_mass_out, void* stream);

/* Effective group count (§5.3): exp(-sum_i a_i log a_i) for the group
 * probabilities a_i = mass_i / sum(mass) (0 log 0 = 0) -- a dispersion
 * measure: n for a uniform spread over n groups, 1 for a single group.
 * mass host [n_groups], non-negative, not all zero; *out host.  Host only.
 * Errors: KVM_E_INVAL. */
kvm_status kvm_effective_group_count(int32_t n_groups, const double* mass, double* out);

/* Total variation distance between two distributions over the same n
 * entries (§6.3): 0.5 * sum_i |p_i - q_i|.  Host only.  Errors: KVM_E_INVAL. */
kvm_status kvm_total_variation(int32_t n, const double* p, const double* q, double* out);

/* Copy the whole state of `src` into `dst`: every character's live KV,
 * positions, recurrent states, live lengths and cursors (§4.2: task-specific
 * continuations branch from a maintained root).  Both contexts must have the
 * same model shape, character count and capacities (max_tail_tokens may
 * differ).  Enqueued on `stream`; dst's previous state is overwritten.
 * Errors: KVM_E_INVAL (shapes differ). */
kvm_status kvm_fork(kvm_ctx* dst, const kvm_ctx* src, void* stream);

/* Per-kernel timing for diagnostics.  While enabled, each kernel launch of
 * the library is bracketed by a pair of CUDA events on its stream.
 * kvm_profile_read synchronizes the device and returns, for one kernel
 * family (KVM_K_*), the number of timed launches and their summed device
 * time in milliseconds since the last reset; reset != 0 clears every family.
 * Events come from a pool made at enable time (4096 launches between
 * reads); launches beyond it are neither timed nor counted here
 * (kvm_launch_count counts every launch). */
enum { KVM_K_COMPACT = 0, KVM_K_ROPE_APPEND = 1, KVM_K_ATTENTION = 2, KVM_K_ATTN_COMBINE = 3,
       KVM_K_GDN = 4, KVM_K_GATHER = 5, KVM_K_GDN_PREP = 6, KVM_K_GDN_CONV = 7, KVM_K_COUNT = 8 };
kvm_status kvm_profile_enable(kvm_ctx* ctx, int32_t enable);
kvm_status kvm_profile_read(kvm_ctx* ctx, int32_t kernel, int64_t* launches, double* total_ms,
                            int32_t reset);

/* Synchronize `stream` and read the device error word; returns KVM_E_DEVICE
 * (and clears the word) if a kernel reported a violation since the last
 * check. */
kvm_status kvm_check(kvm_ctx* ctx, void* stream);

/* Launch plans of the delta-rule layers (no paper counterpart; fused
 * defaults to on, state chain to off).
 * KVM_PLAN_GDN_STATE_CHAIN (d_k = d_v = 128, one or few characters): the
 * serial chunk chain carries only the state, S^T <- P_c S^T + B_c with
 * P_c = G_C I - K^T diag(w) W and B_c = K^T diag(w) U formed in the
 * parallel prep, and the chunks' outputs O = A U + Q' S0^T follow in one
 * parallel pass over per-chunk state snapshots.  Off: the chain also forms
 * E = U - W S0^T and the outputs.  The two forms round differently (both
 * within the library's accuracy).  Measured in a stack of delta-rule layers
 * (1024-token tail): the state chain takes 36 us against 52 for the full
 * chain, but its larger prep and the output pass make a layer 86 us against
 * 60, so it is off by default.
 * KVM_PLAN_GDN_FUSED: when a round has few characters and long tails, the
 * prep and the chain run in one launch, prep blocks publishing each chunk's
 * record through flags to the chain blocks; off: a prep launch, then the
 * chain's.  Bit-identical either way.  If the device refuses the one-launch
 * form, the context uses two launches from then on.
 * Errors: KVM_E_INVAL. */
enum { KVM_PLAN_GDN_FUSED = 0, KVM_PLAN_GDN_STATE_CHAIN = 1 };
kvm_status kvm_set_plan(kvm_ctx* ctx, int32_t what, int32_t enable);

/* Failure-detection hook of the compaction's bounded waits (no paper
 * counterpart).  polls: how many times a compaction block polls an earlier
 * chunk's read flag before it gives up (0 restores the default, ~0.3-1 s).
 * stall != 0: every block of later compactions of this context also waits
 * on a device word that nothing sets, so each gives up after `polls` polls,
 * moves nothing and reports an expired wait, which kvm_check returns as
 * KVM_E_DEVICE (the context's caches are then undefined: restore them, e.g.
 * with kvm_fork from a root).  Tests use it to exercise the failure path
 * without a fault.  Errors: KVM_E_INVAL. */
kvm_status kvm_debug_compact_wait(kvm_ctx* ctx, int32_t polls, int32_t stall);

/* Debug builds (compiled with -DKVM_DEBUG) surround every device buffer of
 * a context with canary bands, which kvm_check verifies (KVM_E_DEVICE names
 * the buffer whose band changed).  This call overwrites one byte just past
 * the context's first buffer, so that tests can exercise that check without
 * a faulty kernel.  Release builds: KVM_E_UNSUPPORTED.  No paper
 * counterpart. */
kvm_status kvm_debug_poke_canary(kvm_ctx* ctx);

/* Number of kernel launches the library has enqueued since creation
 * (diagnostics for the benchmark). */
int64_t kvm_launch_count(const kvm_ctx* ctx);

#ifdef __cplusplus
}
#endif
#endif /* KVM_H */
