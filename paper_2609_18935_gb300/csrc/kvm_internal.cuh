// Internal declarations of the maintenance library (kernels + host runtime).
// Everything here is private to libkvm; the public ABI is include/kvm.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace kvm {

// Programmatic dependent launch: every kernel of the library is launched so
// that it may start while the previous kernel of the stream finishes.  A
// kernel calls grid_dependency_wait() before its first global memory access
// (it returns once the previous grid has completed and its writes are
// visible), so stream order is kept; grid_dependents_launch() then lets the
// next kernel's blocks be scheduled and run their prologue early.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dependents_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename Params>
inline cudaError_t launch_pdl(void (*kernel)(Params), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              const Params& p) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, p);
}

constexpr int kMaxChars = 256;      // characters per context (per-round descriptors travel as kernel parameters)
constexpr int kMaxSpans = 1024;     // deletion spans per round, all characters together
constexpr int kMaxRotaryHalf = 128; // rotary_dim / 2

// Device error word bits (read by kvm_check).
constexpr int kErrBounds = 1;       // an index fell outside the buffers a kernel was given
constexpr int kErrWait = 2;         // a bounded wait expired

// ----------------------------------------------------------------------------
// kv_compact
// ----------------------------------------------------------------------------
constexpr int kCompactThreads = 256;
constexpr int kCompactVecPerThread = 8;            // 16-byte vectors held per thread (8: 418 us against 531 with 4 for the 1.5 GB of the 48-layer round)
constexpr int kCompactVecPerChunk = kCompactThreads * kCompactVecPerThread;
constexpr int kCompactWaitLimit = 1 << 22;        // default polls of a read flag (~0.3-1 s with the back-off)

struct CompactChar {
    int32_t L_new;        // live length after removal
    int32_t first;        // first removed live index (= first moved destination)
    int32_t seg_off;      // offset of this character's segments in seg_start/seg_shift
    int32_t n_seg;        // number of spans (= moved segments)
    int32_t cap_off;      // slot offset of the character inside every slab
    int32_t chunks_kv;    // chunks per KV slab
    int32_t chunks_pos;   // chunks of the position slab
    int32_t blk_off;      // first block of this character
    int32_t flag_off;     // first read-flag of this character
};

struct CompactParams {
    int32_t n_chars;
    int32_t n_kv_slabs;   // 2 * n_attn * n_kv_heads  (K slabs, then V slabs)
    int32_t vec_per_row;  // 16-byte vectors per KV row (head_dim * 2 / 16)
    int32_t rows_kv;      // rows per KV chunk
    int32_t rows_pos;     // rows per position chunk
    int32_t total_blocks;
    uint32_t epoch;
    int64_t slab_rows;    // rows per (layer, head) slab = total capacity
    uint4* K;
    uint4* V;
    int32_t* pos;
    int32_t* tickets;     // [n_chars][n_kv_slabs + 1]
    uint32_t* flags;      // read flag of chunk i at flags[i * flag_stride]
    int32_t flag_stride;  // 32 keeps every flag in its own 128-byte line (no line shared by pollers)
    int32_t* err;
    int32_t wait_limit;   // polls of a read flag before the wait gives up (kErrWait)
    // failure-detection test only: when set, every block also waits on this
    // word, which nothing ever sets, so its wait expires after wait_limit polls
    const uint32_t* never_set;
    CompactChar ch[kMaxChars];
    // segment k of a character: survivors whose new index is >= seg_start[k]
    // (and below the next segment's start) come from new index + seg_shift[k]
    int32_t seg_start[kMaxSpans];
    int32_t seg_shift[kMaxSpans];
};

void launch_kv_compact(const CompactParams& p, cudaStream_t s);

struct GatherParams {
    int32_t n_chars;
    int32_t total;        // sum of L_new
    int32_t out_off[kMaxChars + 1];
    int32_t first[kMaxChars];
    int32_t seg_off[kMaxChars];
    int32_t n_seg[kMaxChars];
    int32_t* out;
    int32_t seg_start[kMaxSpans];
    int32_t seg_shift[kMaxSpans];
};
void launch_gather_map(const GatherParams& p, cudaStream_t s);

// ----------------------------------------------------------------------------
// tail attention
// ----------------------------------------------------------------------------
struct AttnChar {
    int32_t L_prev;       // surviving live entries (L')
    int32_t M;            // tail tokens
    int32_t tail_off;     // first packed tail row
    int32_t cap_off;      // slot offset of the character in the slabs
    int64_t p;            // cursor: position of tail token 0
    int32_t n_qtiles;     // query tiles per KV head
    int32_t tile_off;     // first query tile of this character (tiles ordered character, KV head, tile)
};

// The attention's work is the list of (query tile, 64-key tile) units, query
// tiles in order and each tile's key tiles in order; persistent block c
// processes units [start_c, start_{c+1}), given as (query tile, key tile).
constexpr int kMaxAttnCtas = 320;

struct AttnParams {
    // TMA maps: every layer's K / V slabs as rows of D (box 64 x 64), 128-byte swizzle
    CUtensorMap tmap_k;
    CUtensorMap tmap_v;
    int32_t attn_layer;   // index among attention layers
    int32_t n_chars;
    int32_t Hq, Hkv, D, R, g;
    int32_t n_tiles;      // query tiles over all characters and KV heads
    int32_t n_ctas;       // persistent attention blocks
    int32_t tok_per_tile; // tail tokens per 128-row query tile (128 / g)
    float scale_log2;     // log2(e) / sqrt(D)
    int64_t slab_rows;    // rows per (layer, head) slab
    const __nv_bfloat16* q;       // caller's unrotated q  [sum M][Hq][D]
    const __nv_bfloat16* k_new;   // [sum M][Hkv][D]
    const __nv_bfloat16* v_new;
    __nv_bfloat16* q_rot;         // workspace [sum M][Hq][D]
    __nv_bfloat16* K;             // this layer's K slabs [Hkv][slab_rows][D]
    __nv_bfloat16* V;
    int32_t* pos;                 // [slab_rows]
    __nv_bfloat16* out;           // [sum M][Hq][D]
    const int32_t* tail_pos;      // device [sum M] position of each tail token, or null: p + i
    float* part_o;                // [2 n_ctas][D / 32][8][128][4]: partial O of a block's first / last segment
    float* part_ml;               // [2 n_ctas][128][2]: (reference max in log2 units, sum) of a partial
    int32_t* err;
    int32_t* diag;                // first expired wait: block + 1, tag, parity
    double inv_freq[kMaxRotaryHalf];
    int32_t cta_tile[kMaxAttnCtas + 1];
    int32_t cta_k[kMaxAttnCtas + 1];
    int32_t n_split_tiles;                   // query tiles shared by several blocks
    int32_t split_cb[kMaxAttnCtas];          // per such tile: the first block that starts inside it
    AttnChar ch[kMaxChars];
};

void launch_rope_append(const AttnParams& p, int total_tokens, cudaStream_t s);

// Key re-rotation (tail-and-relocate, §5.2): rotate stored keys of live slots
// [slot0, slot0 + n) in every attention layer by (new_pos - pos), then set pos.
struct RerotateParams {
    int32_t n;            // entries
    int32_t n_attn, Hkv, D, R;
    int64_t slot0;        // first slot (character offset + live index)
    int64_t slab_rows;
    __nv_bfloat16* K;     // all layers' K slabs [n_attn][Hkv][slab_rows][D]
    int32_t* pos;         // [slab_rows]
    const int32_t* new_pos;   // device [n]
    int32_t* err;
    double inv_freq[kMaxRotaryHalf];
};
void launch_rerotate(const RerotateParams& p, cudaStream_t s);
void launch_tail_attention(const AttnParams& p, cudaStream_t s);
void launch_attn_combine(const AttnParams& p, cudaStream_t s);
int attention_ctas_per_sm(int head_dim);
constexpr int kAttnRows = 128;   // query rows per attention tile

// ----------------------------------------------------------------------------
// attention-probe diagnostics (§5.3, Appendix C)
// ----------------------------------------------------------------------------
constexpr int kProbeMaxQueries = 16;   // probe queries per call (the paper averages the last 8)
constexpr int kProbeKeys = 64;         // keys per probe block

struct ProbeParams {
    int32_t L;            // live entries of the character
    int32_t n_q;          // probe queries: the last n_q live entries
    int32_t Hq, Hkv, D, R, g;
    int32_t n_groups;
    float scale;          // 1 / sqrt(D)
    int64_t slab_rows;
    int64_t slot0;        // the character's first slot
    const __nv_bfloat16* q;   // caller's unrotated probe queries [n_q][Hq][D]
    float* q_rot;             // workspace [n_q][Hq][D] fp32
    const __nv_bfloat16* K;   // this layer's K slabs [Hkv][slab_rows][D]
    const int32_t* pos;       // [slab_rows]
    float* part;              // workspace [ceil(L / 64)][n_q * Hq][2]: per key tile (max, sum)
    float* row_ms;            // workspace [n_q * Hq][2]: per query row (max, sum)
    float* probs;             // out [L]
    const int32_t* group_of;  // [L] or null
    float* group_mass;        // out [n_groups]
    int32_t* err;
    double inv_freq[kMaxRotaryHalf];
};
void launch_attn_probe(const ProbeParams& p, cudaStream_t s);

// ----------------------------------------------------------------------------
// gated delta rule
// ----------------------------------------------------------------------------
struct GdnChar {
    int32_t M;
    int32_t tail_off;
    int32_t chunk_off;        // first 64-token chunk of this character (all characters' chunks numbered in order)
};

struct GdnParams {
    int32_t n_chars, H, dk, dv;
    int32_t dv_slice;         // rows of S per block (a multiple of 16, <= 128, dividing dv)
    int32_t prep_parts;       // prep blocks per (chunk, head): 1, or 2 (one writes [W; Q'] and K, one U | A U)
    const __nv_bfloat16* q;   // [sum M][H][dk]
    const __nv_bfloat16* k;
    const __nv_bfloat16* v;   // [sum M][H][dv]
    const float* alpha;       // [sum M][H]
    const float* beta;
    __nv_bfloat16* out;       // [sum M][H][dv]
    float* S;                 // this layer's state [n_chars][H][dv][dk]
    uint8_t* work;            // per (chunk, head) records written by the prep pass, read by the scan
    int64_t rec_bytes;        // bytes per record
    int32_t total_chunks;     // sum over characters of ceil(M / 64)
    int32_t* err;
    int32_t* diag;            // first expired wait: block + 1, tag, parity
    // fused launches (launch_gdn_fused): the first n_scan blocks are scan
    // items, the rest prep workers; record r is published by flags[32 r] = epoch
    int32_t n_scan;
    uint32_t epoch;
    uint32_t* flags;
    // v2: the state entering each chunk, per (chunk, head), as the output pass reads it
    uint8_t* snap;
    int64_t snap_bytes;
    GdnChar ch[kMaxChars];
};

// Short convolution (width 4) + SiLU of a delta-rule layer's q/k/v with the
// carried conv state; k is L2-normalised per head afterwards.
struct ConvParams {
    int32_t n_chars, H, dk, dv, channels;     // channels = H (2 d_k + d_v)
    int32_t total;                            // sum M
    int32_t tail_cu[kMaxChars + 1];
    const __nv_bfloat16* xq;                  // caller's pre-conv inputs [sum M][H][d_k]
    const __nv_bfloat16* xk;
    const __nv_bfloat16* xv;                  // [sum M][H][d_v]
    const float* w;                           // [channels][4]
    const __nv_bfloat16* state_in;            // [n_chars][3][channels]: the last 3 inputs before the tail
    __nv_bfloat16* state_out;                 // [n_chars][3][channels]: the last 3 inputs after it
    __nv_bfloat16* yq;                        // outputs, laid out like the inputs
    __nv_bfloat16* yk;
    __nv_bfloat16* yv;
    int32_t* err;
};
void launch_gdn_conv(const ConvParams& p, cudaStream_t s);

// Bytes of one (chunk, head) record of the delta-rule workspace.
int64_t gdn_record_bytes(int dk, int dv);
void launch_gdn_chunk_prep(const GdnParams& p, cudaStream_t s);   // state-independent chunk products
void launch_gdn_chunk_scan(const GdnParams& p, cudaStream_t s);   // chunks in order, state in TMEM
// Both in one launch of `grid` blocks (one per SM at most); returns the
// launch's error (the caller falls back to the two launches).
cudaError_t launch_gdn_fused(const GdnParams& p, int grid, cudaStream_t s);
// v2 (d_k = 128, 32-row slices): prep, state chain and output pass (or, with
// fused_grid > 0, prep and chain in one launch of fused_grid blocks, then the
// output pass).  Returns a refused launch's error before enqueuing anything else.
int64_t gdn_snapshot_bytes(int dk, int dv);
cudaError_t launch_gdn_v2(const GdnParams& p, int fused_grid, cudaStream_t s);

// Set the text returned by kvm_last_error() and return `code`.
int report_error(int code, const char* msg);

}  // namespace kvm
