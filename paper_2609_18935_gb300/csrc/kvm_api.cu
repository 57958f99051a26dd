// Host runtime and C ABI of the maintenance library (include/kvm.h).
//
// The context owns a character population's state (A_t, R_t, p_t) (§4.1):
//   K, V    [n_attn][Hkv][T_cap][D] bf16   (character b at slot offset cap_off[b])
//   pos     [T_cap] int32                  (shared by every attention layer)
//   S       [n_gdn][B][H][d_v][d_k] fp32
//   cursor, live length and a host mirror of positions per character.
// Every argument and span is validated here before anything is enqueued, so a
// rejected call leaves the state untouched.  Per-round descriptors travel to
// the kernels as kernel parameters: nothing is allocated or uploaded per call.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "../../include/kvm.h"
#include "kvm_internal.cuh"
#include "tma_host.h"

using namespace kvm;

namespace {

thread_local std::string g_err;

kvm_status fail(kvm_status code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

#define CUDA_TRY(expr)                                                                  \
    do {                                                                                \
        cudaError_t e_ = (expr);                                                        \
        if (e_ != cudaSuccess)                                                          \
            return fail(KVM_E_CUDA, "%s failed: %s", #expr, cudaGetErrorString(e_));     \
    } while (0)

#define LAUNCH_CHECK(ctx)                                                                \
    do {                                                                                 \
        cudaError_t e_ = cudaGetLastError();                                             \
        if (e_ != cudaSuccess) return fail(KVM_E_CUDA, "kernel launch failed: %s", cudaGetErrorString(e_)); \
    } while (0)

// Persistent attention blocks of a context: one wave on this device, at most
// kMaxAttnCtas.
int attention_grid_cap(int num_sms, int head_dim) {
    return std::max(1, std::min(kMaxAttnCtas, num_sms * attention_ctas_per_sm(head_dim)));
}
constexpr int kMinUnitsPerCta = 4;  // smallest share of (query tile, key tile) units per attention block
constexpr double kSegmentCost = 8.0; // extra cost, in 64-key units, of each segment an attention block starts
constexpr int kFlagStride = 32;     // compaction read flags: one per 128-byte line
constexpr int kMinPrepWorkers = 24; // fused delta-rule launches leave at least this many SMs to the prep

}  // namespace

struct kvm_ctx {
    int device = 0;
    int num_sms = 0;
    // model
    int n_layers = 0;
    std::vector<int> kind, attn_idx, gdn_idx;
    int n_attn = 0, n_gdn = 0;
    int Hq = 0, Hkv = 0, D = 0, R = 0, g = 0;
    double theta = 0;
    int H = 0, dk = 0, dv = 0;
    int conv = 0;                         // short-convolution width of the delta-rule layers (0 or 4)
    int conv_ch = 0;                      // its channels, H (2 d_k + d_v)
    // population
    int B = 0;
    std::vector<int> cap, cap_off;
    int64_t T_cap = 0;
    int max_tail = 0;
    std::vector<int> live;
    std::vector<int64_t> cursor;
    std::vector<std::vector<int32_t>> hpos;
    // device state
    __nv_bfloat16* K = nullptr;
    __nv_bfloat16* V = nullptr;
    int32_t* pos = nullptr;
    float* S = nullptr;
    // workspace
    __nv_bfloat16* q_rot = nullptr;
    // per-token positions (tail placement variants) and re-rotation targets:
    // host values go through a pinned staging buffer, guarded by ev_pos
    int32_t* tail_pos_dev = nullptr;      // [max_tail]
    int32_t* reloc_pos_dev = nullptr;     // [max capacity]
    int32_t* pos_host = nullptr;          // pinned [max(max_tail, max capacity)]
    cudaEvent_t ev_pos = nullptr;
    int max_cap = 0;
    // attention-probe workspace: rotated probe queries, per-tile and per-row softmax partials
    // short convolution: weights [n_gdn][C][4] fp32; state, two buffers per
    // layer [2][n_gdn][B][3][C] bf16 (a round reads one, writes the other,
    // conv_par[layer] tells which is current); outputs [max_tail][H][...] bf16
    float* conv_w = nullptr;
    __nv_bfloat16* conv_state = nullptr;
    std::vector<int> conv_par;
    __nv_bfloat16* conv_y = nullptr;
    float* probe_q = nullptr;
    float* probe_part = nullptr;
    float* probe_rows = nullptr;
    float* part_o = nullptr;
    float* part_ml = nullptr;
    int32_t* tickets = nullptr;
    uint32_t* flags = nullptr;
    std::vector<int> flag_off;
    uint32_t epoch = 0;
    int32_t* err = nullptr;
    int32_t* diag = nullptr;              // [16]: where the first expired device wait gave up
    uint8_t* gdn_work = nullptr;          // delta-rule prep records
    int64_t gdn_rec = 0;
    // fused prep + scan launches: per-record flags (128-byte lines) and the
    // launch epoch they are compared with; gdn_fuse off = always two launches
    uint32_t* gdn_flags = nullptr;
    uint32_t gdn_epoch = 0;
    bool gdn_fuse = true;
    // state-chain form (d_k = d_v = 128): per-chunk snapshots of the state
    uint8_t* gdn_snap = nullptr;
    int64_t gdn_snap_bytes = 0;
    bool gdn_chain = false;
    // staging for host-resident rounds: every layer's inputs (q, k, v, alpha,
    // beta) and output have their own buffers, so the copies of all layers
    // run on a copy stream beside the kernels
    uint8_t* stage = nullptr;
    std::vector<size_t> stage_in_off;     // [n_layers * 5]
    std::vector<size_t> stage_out_off;    // [n_layers]
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t ev_start = nullptr, ev_copies = nullptr;
    // a round's compaction runs on its own stream beside the recurrent layers
    // that come before the first attention layer (it touches only the KV cache)
    cudaStream_t compact_stream = nullptr;
    cudaEvent_t ev_round = nullptr, ev_compacted = nullptr;
    // per attention layer: the main stream reached the layers its compaction
    // runs beside, and that compaction is done
    std::vector<cudaEvent_t> ev_piece_go, ev_piece_done;
    std::vector<cudaEvent_t> ev_in, ev_done;   // per layer: inputs landed, outputs written
    double inv_freq[kMaxRotaryHalf] = {};
    CUtensorMap tmap_k, tmap_v;           // TMA maps of K, V (attention layers only)
    int64_t launches = 0;
    int rows_kv = 0, rows_pos = 0;
    int compact_wait_limit = kCompactWaitLimit;   // polls of a compaction read flag before giving up
    bool compact_stall = false;                   // failure-detection tests: wait on a word nothing sets
    // every device buffer the context owns: allocation base, user bytes, name
    // (with KVM_DEBUG the user bytes sit between two canary bands)
    struct DevAlloc { void* base; size_t bytes; const char* name; };
    std::vector<DevAlloc> allocs;
    // per-kernel timing (kvm_profile_*)
    bool prof = false;
    std::vector<cudaEvent_t> ev;          // 2 per timed launch
    std::vector<int> ev_kind;             // kind of each recorded pair
};

namespace {

// Debug builds (-DKVM_DEBUG) put a band of kCanaryByte before and after
// every device buffer of a context; kvm_check reads the bands back and
// reports a kernel that wrote outside its buffers as KVM_E_DEVICE.
#ifdef KVM_DEBUG
constexpr size_t kCanary = 4096;        // keeps the user pointer 256-byte aligned
#else
constexpr size_t kCanary = 0;
#endif
constexpr unsigned char kCanaryByte = 0xA5;

// One device buffer of `count` T, zeroed (or not), registered for release
// and for the canary check.
template <typename T>
cudaError_t alloc_dev(kvm_ctx* c, T** p, size_t count, const char* name, bool zero = true) {
    *p = nullptr;
    if (count == 0) return cudaSuccess;
    const size_t bytes = count * sizeof(T);
    void* base = nullptr;
    cudaError_t e = cudaMalloc(&base, bytes + 2 * kCanary);
    if (e != cudaSuccess) return e;
    c->allocs.push_back({base, bytes, name});
    char* user = static_cast<char*>(base) + kCanary;
    if (kCanary) {
        e = cudaMemset(base, kCanaryByte, kCanary);
        if (e == cudaSuccess) e = cudaMemset(user + bytes, kCanaryByte, kCanary);
        if (e != cudaSuccess) return e;
    }
    *p = reinterpret_cast<T*>(user);
    return zero ? cudaMemset(user, 0, bytes) : cudaSuccess;
}

#define alloc_zero(pp, count) alloc_dev(c, pp, count, #pp)

void free_all(kvm_ctx* c) {
    for (const auto& a : c->allocs) cudaFree(a.base);
    c->allocs.clear();
    if (c->pos_host) cudaFreeHost(c->pos_host);
    if (c->ev_pos) cudaEventDestroy(c->ev_pos);
    for (cudaEvent_t e : c->ev_in) if (e) cudaEventDestroy(e);
    for (cudaEvent_t e : c->ev_done) if (e) cudaEventDestroy(e);
    if (c->ev_start) cudaEventDestroy(c->ev_start);
    if (c->ev_copies) cudaEventDestroy(c->ev_copies);
    if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
    if (c->ev_round) cudaEventDestroy(c->ev_round);
    if (c->ev_compacted) cudaEventDestroy(c->ev_compacted);
    for (cudaEvent_t e : c->ev_piece_go) if (e) cudaEventDestroy(e);
    for (cudaEvent_t e : c->ev_piece_done) if (e) cudaEventDestroy(e);
    if (c->compact_stream) cudaStreamDestroy(c->compact_stream);
    for (cudaEvent_t e : c->ev) cudaEventDestroy(e);
    c->ev.clear();
}

kvm_status check_tail_cu(const kvm_ctx* c, const int32_t* tail_cu, int* total) {
    if (!tail_cu) return fail(KVM_E_INVAL, "tail_cu is NULL");
    if (tail_cu[0] != 0) return fail(KVM_E_INVAL, "tail_cu[0] must be 0");
    for (int b = 0; b < c->B; ++b) {
        const int m = tail_cu[b + 1] - tail_cu[b];
        if (m < 0) return fail(KVM_E_INVAL, "tail_cu not monotone at character %d", b);
    }
    *total = tail_cu[c->B];
    if (*total > c->max_tail)
        return fail(KVM_E_CAPACITY, "sum M = %d exceeds max_tail_tokens = %d", *total, c->max_tail);
    return KVM_OK;
}

kvm_status check_layer(const kvm_ctx* c, int layer, int want) {
    if (layer < 0 || layer >= c->n_layers) return fail(KVM_E_INVAL, "layer %d out of range", layer);
    if (c->kind[layer] != want)
        return fail(KVM_E_INVAL, "layer %d is not a %s layer", layer,
                    want == KVM_LAYER_ATTN ? "attention" : "delta-rule");
    return KVM_OK;
}

constexpr int kProfPool = 4096;

// Bracket one launch with a pair of events when profiling is on.
int prof_begin(kvm_ctx* c, int kind, cudaStream_t s) {
    ++c->launches;
    if (!c->prof) return -1;
    const int slot = (int)c->ev_kind.size();
    if (slot >= kProfPool) return -1;
    c->ev_kind.push_back(kind);
    cudaEventRecord(c->ev[2 * slot], s);
    return slot;
}

void prof_end(kvm_ctx* c, int slot, cudaStream_t s) {
    if (slot >= 0) cudaEventRecord(c->ev[2 * slot + 1], s);
}

// Copy n host positions into the device buffer dev on stream s through the
// context's pinned staging buffer (the previous staging copy must have left
// it first, which ev_pos tracks).
kvm_status stage_positions(kvm_ctx* c, const int32_t* host, int n, int32_t* dev, cudaStream_t s) {
    if (n <= 0) return KVM_OK;
    CUDA_TRY(cudaEventSynchronize(c->ev_pos));
    std::memcpy(c->pos_host, host, sizeof(int32_t) * (size_t)n);
    CUDA_TRY(cudaMemcpyAsync(dev, c->pos_host, sizeof(int32_t) * (size_t)n, cudaMemcpyHostToDevice, s));
    CUDA_TRY(cudaEventRecord(c->ev_pos, s));
    return KVM_OK;
}

// Per-token positions, if given, must be non-negative (they are int32, so
// no id passes 2^31 - 1); without them the cursor must leave room for M ids.
kvm_status check_positions(const kvm_ctx* c, const int32_t* tail_cu, const int32_t* tail_pos) {
    for (int b = 0; b < c->B; ++b) {
        const int m = tail_cu[b + 1] - tail_cu[b];
        if (tail_pos) {
            for (int i = tail_cu[b]; i < tail_cu[b + 1]; ++i)
                if (tail_pos[i] < 0) return fail(KVM_E_INVAL, "character %d: tail position %d is negative", b, i);
        } else if (c->cursor[b] + m > INT32_MAX) {
            return fail(KVM_E_CAPACITY, "character %d: position ids overflow", b);
        }
    }
    return KVM_OK;
}

// Validate one round's spans and build the per-character segment tables.
struct SpanPlan {
    std::vector<int> L_new, first, seg_off, n_seg;
    std::vector<int32_t> seg_start, seg_shift;
};

// B characters with live lengths live[B] (host state, no device access).
kvm_status plan_spans_for(int B, const int* live, const int32_t* span_cu, const int32_t* sb, const int32_t* se,
                          SpanPlan& pl) {
    if (!span_cu) return fail(KVM_E_INVAL, "span_cu is NULL");
    if (span_cu[0] != 0) return fail(KVM_E_INVAL, "span_cu[0] must be 0");
    const int total = span_cu[B];
    if (total < 0) return fail(KVM_E_INVAL, "negative span count");
    if (total > kMaxSpans) return fail(KVM_E_INVAL, "%d spans exceed the per-round limit %d", total, kMaxSpans);
    if (total > 0 && (!sb || !se)) return fail(KVM_E_INVAL, "span arrays are NULL");
    pl.L_new.assign(B, 0);
    pl.first.assign(B, 0);
    pl.seg_off.assign(B, 0);
    pl.n_seg.assign(B, 0);
    pl.seg_start.clear();
    pl.seg_shift.clear();
    for (int b = 0; b < B; ++b) {
        const int s0 = span_cu[b], s1 = span_cu[b + 1];
        if (s1 < s0 || s0 < 0 || s1 > total)
            return fail(KVM_E_INVAL, "span_cu not monotone at character %d", b);
        const int L = live[b];
        int removed = 0, prev_end = 0;
        pl.seg_off[b] = (int)pl.seg_start.size();
        pl.n_seg[b] = s1 - s0;
        for (int k = s0; k < s1; ++k) {
            const int lo = sb[k], hi = se[k];
            if (!(0 <= lo && lo < hi && hi <= L))
                return fail(KVM_E_SPAN, "character %d span %d [%d,%d) empty or outside live [0,%d)", b, k - s0,
                            lo, hi, L);
            if (k > s0 && lo < prev_end)
                return fail(KVM_E_SPAN, "character %d span %d overlaps or precedes the previous span", b, k - s0);
            prev_end = hi;
            removed += hi - lo;
            // survivors after this span: new index (hi - removed) onward come from + removed
            pl.seg_start.push_back(hi - removed);
            pl.seg_shift.push_back(removed);
        }
        pl.L_new[b] = L - removed;
        pl.first[b] = (s1 > s0) ? sb[s0] : pl.L_new[b];
    }
    return KVM_OK;
}

kvm_status plan_spans(const kvm_ctx* c, const int32_t* span_cu, const int32_t* sb, const int32_t* se,
                      SpanPlan& pl) {
    return plan_spans_for(c->B, c->live.data(), span_cu, sb, se, pl);
}

// The attention's work partition for one layer: query tiles numbered
// (character, KV head, tile), each with the 64-key tiles it attends to
// (every surviving entry plus the tail up to its last token).  Stream-K with
// a cost model: block cc gets a contiguous range of (query tile, key tile)
// units; a unit costs 1 and every segment a block starts (its first one, and
// each query tile it enters) costs kSegmentCost more (Q staging, the
// epilogue, the pipeline refill).  The ranges are cut greedily at a
// per-block cost target, found by bisection so that exactly G blocks cover
// the units with the least maximum cost.  Tiles shared by several blocks are
// merged once, from the first block that starts inside them (split_cb).
struct AttnPlan {
    int n_tiles = 0, n_ctas = 0;
    std::vector<int> n_qtiles, tile_off;             // per character
    std::vector<int32_t> cta_tile, cta_k, split_cb;  // [n_ctas + 1], [n_ctas + 1], [number of split tiles]
};

void plan_attention(int B, const int* L_prev, const int* M, int Hkv, int tpt, int grid_cap, AttnPlan& pl) {
    pl.n_qtiles.assign(B, 0);
    pl.tile_off.assign(B, 0);
    std::vector<int> nk_of;
    int tiles = 0;
    int64_t units = 0;
    for (int b = 0; b < B; ++b) {
        pl.n_qtiles[b] = (M[b] + tpt - 1) / tpt;
        pl.tile_off[b] = tiles;
        tiles += Hkv * pl.n_qtiles[b];
    }
    nk_of.reserve(tiles);
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < Hkv; ++h)
            for (int qt = 0; qt < pl.n_qtiles[b]; ++qt) {
                nk_of.push_back((L_prev[b] + std::min(M[b], (qt + 1) * tpt) + 63) / 64);
                units += nk_of.back();
            }
    pl.n_tiles = tiles;
    const int G = (int)std::max<int64_t>(1, std::min<int64_t>(grid_cap, units / kMinUnitsPerCta));
    pl.n_ctas = G;
    pl.cta_tile.assign(G + 1, 0);
    pl.cta_k.assign(G + 1, 0);
    // blocks needed to cover everything with ranges of cost <= target; the
    // cut points go to cta_tile / cta_k when `emit`
    auto cover = [&](double target, bool emit) -> int {
        int blocks = 1;
        double cost = kSegmentCost;
        for (int t = 0; t < (int)nk_of.size(); ++t) {
            int k = 0;
            if (t > 0) cost += kSegmentCost;                  // entering a new query tile
            while (k < nk_of[t]) {
                const double room = target - cost;
                const int take = room >= nk_of[t] - k ? nk_of[t] - k : std::max(0, (int)room);
                k += take;
                cost += take;
                if (k < nk_of[t] && (take == 0 || cost >= target)) {
                    if (take == 0 && cost == kSegmentCost) {      // a block must take at least a unit
                        ++k;
                        cost += 1;
                        if (k >= nk_of[t]) break;
                    }
                    if (emit && blocks <= G) { pl.cta_tile[blocks] = t; pl.cta_k[blocks] = k; }
                    ++blocks;
                    cost = kSegmentCost;
                }
            }
        }
        return blocks;
    };
    double lo = (double)units / G, hi = (double)units / G + 2.0 * kSegmentCost * (1 + tiles / G) + 1.0;
    while (cover(hi, false) > G) hi *= 2;
    for (int it = 0; it < 40 && hi - lo > 0.25; ++it) {
        const double mid = 0.5 * (lo + hi);
        if (cover(mid, false) <= G) hi = mid; else lo = mid;
    }
    const int used = cover(hi, true);
    // fewer ranges than blocks: the spare blocks get empty ranges at the end
    for (int cc = used; cc <= G; ++cc) { pl.cta_tile[cc] = tiles; pl.cta_k[cc] = 0; }
    pl.split_cb.clear();
    for (int cc = 1; cc < G; ++cc)
        if (pl.cta_k[cc] > 0 && !(pl.cta_tile[cc - 1] == pl.cta_tile[cc] && pl.cta_k[cc - 1] > 0))
            pl.split_cb.push_back(cc);
}

}  // namespace

// ============================================================================
// lifetime
// ============================================================================
extern "C" kvm_status kvm_create(const kvm_model_desc* m, int32_t n_chars, const int32_t* capacity,
                                 int32_t max_tail_tokens, kvm_ctx** out) {
    if (!m || !capacity || !out) return fail(KVM_E_INVAL, "NULL argument");
    *out = nullptr;
    if (m->n_layers <= 0 || !m->layer_kind) return fail(KVM_E_INVAL, "model has no layers");
    if (n_chars <= 0 || n_chars > kMaxChars) return fail(KVM_E_INVAL, "n_chars must be in [1,%d]", kMaxChars);
    if (max_tail_tokens <= 0) return fail(KVM_E_INVAL, "max_tail_tokens must be positive");
    kvm_ctx* c = new kvm_ctx();
    c->n_layers = m->n_layers;
    for (int l = 0; l < m->n_layers; ++l) {
        const int k = m->layer_kind[l];
        if (k != KVM_LAYER_ATTN && k != KVM_LAYER_GDN) { delete c; return fail(KVM_E_INVAL, "bad layer kind"); }
        c->kind.push_back(k);
        c->attn_idx.push_back(k == KVM_LAYER_ATTN ? c->n_attn++ : -1);
        c->gdn_idx.push_back(k == KVM_LAYER_GDN ? c->n_gdn++ : -1);
    }
    if (c->n_attn > 0) {
        c->Hq = m->n_q_heads; c->Hkv = m->n_kv_heads; c->D = m->head_dim; c->R = m->rotary_dim;
        c->theta = m->rope_theta;
        if (c->Hkv <= 0 || c->Hq <= 0 || c->Hq % c->Hkv) { delete c; return fail(KVM_E_UNSUPPORTED, "n_q_heads must be a multiple of n_kv_heads"); }
        c->g = c->Hq / c->Hkv;
        if (c->g > 64 || (c->g & (c->g - 1))) { delete c; return fail(KVM_E_UNSUPPORTED, "group size must be a power of two <= 64"); }
        if (c->D != 64 && c->D != 128 && c->D != 256) { delete c; return fail(KVM_E_UNSUPPORTED, "head_dim must be 64, 128 or 256"); }
        if (c->R < 0 || c->R > c->D || (c->R & 1)) { delete c; return fail(KVM_E_UNSUPPORTED, "rotary_dim must be even and <= head_dim"); }
        if (!(c->theta > 0)) { delete c; return fail(KVM_E_INVAL, "rope_theta must be positive"); }
        for (int d = 0; d < c->R / 2; ++d) c->inv_freq[d] = std::pow(c->theta, -2.0 * d / c->R);
    }
    if (c->n_gdn > 0) {
        c->H = m->n_gdn_heads; c->dk = m->d_k; c->dv = m->d_v;
        if (c->H <= 0) { delete c; return fail(KVM_E_INVAL, "n_gdn_heads must be positive"); }
        if (c->dk != 64 && c->dk != 128) { delete c; return fail(KVM_E_UNSUPPORTED, "d_k must be 64 or 128"); }
        if (c->dv <= 0 || c->dv % 32 || c->dv > 128) { delete c; return fail(KVM_E_UNSUPPORTED, "d_v must be a multiple of 32, <= 128"); }
        if (m->conv_kernel != 0 && m->conv_kernel != 4) { delete c; return fail(KVM_E_UNSUPPORTED, "conv_kernel must be 0 or 4"); }
        c->conv = m->conv_kernel;
        c->conv_ch = c->H * (2 * c->dk + c->dv);
    } else if (m->conv_kernel != 0 && m->conv_kernel != 4) {
        delete c;
        return fail(KVM_E_UNSUPPORTED, "conv_kernel must be 0 or 4");
    }
    c->B = n_chars;
    c->max_tail = max_tail_tokens;
    for (int b = 0; b < n_chars; ++b) {
        if (capacity[b] <= 0) { delete c; return fail(KVM_E_INVAL, "capacity of character %d must be positive", b); }
        const int cp = (capacity[b] + 63) / 64 * 64;   // slab offsets stay 64-row aligned
        c->cap.push_back(cp);
        c->cap_off.push_back((int)c->T_cap);
        c->T_cap += cp;
    }
    if (c->T_cap > INT32_MAX) { delete c; return fail(KVM_E_CAPACITY, "total capacity too large"); }
    c->live.assign(n_chars, 0);
    c->cursor.assign(n_chars, 0);
    c->hpos.assign(n_chars, {});

    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) { delete c; return fail(KVM_E_CUDA, "no CUDA device: %s", cudaGetErrorString(e)); }

    const size_t kv_elems = (size_t)c->n_attn * c->Hkv * c->T_cap * c->D;
    const int vec_per_row = c->D * 2 / 16;
    c->rows_kv = c->n_attn ? kCompactVecPerChunk / std::max(vec_per_row, 1) : 1;
    c->rows_pos = kCompactVecPerChunk;
    const int n_kv_slabs = 2 * c->n_attn * c->Hkv;
    size_t n_flags = 0;
    for (int b = 0; b < n_chars; ++b) {
        c->flag_off.push_back((int)n_flags);
        n_flags += (size_t)n_kv_slabs * ((c->cap[b] + c->rows_kv - 1) / c->rows_kv) +
                   (c->cap[b] + c->rows_pos - 1) / c->rows_pos;
    }
    e = cudaSuccess;
    if (e == cudaSuccess) e = alloc_zero(&c->K, kv_elems);
    if (e == cudaSuccess) e = alloc_zero(&c->V, kv_elems);
    if (e == cudaSuccess) e = alloc_zero(&c->pos, c->n_attn ? (size_t)c->T_cap : 0);
    if (e == cudaSuccess) e = alloc_zero(&c->S, (size_t)c->n_gdn * n_chars * c->H * c->dv * c->dk);
    if (e == cudaSuccess) e = alloc_zero(&c->q_rot, c->n_attn ? (size_t)max_tail_tokens * c->Hq * c->D : 0);
    for (int b = 0; b < n_chars; ++b) c->max_cap = std::max(c->max_cap, c->cap[b]);
    if (e == cudaSuccess) e = alloc_zero(&c->tail_pos_dev, c->n_attn ? (size_t)max_tail_tokens : 0);
    if (e == cudaSuccess) e = alloc_zero(&c->reloc_pos_dev, c->n_attn ? (size_t)c->max_cap : 0);
    if (e == cudaSuccess && c->n_attn)
        e = cudaHostAlloc(reinterpret_cast<void**>(&c->pos_host),
                          sizeof(int32_t) * std::max(max_tail_tokens, c->max_cap), cudaHostAllocDefault);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_pos, cudaEventDisableTiming);
    if (c->conv) {
        c->conv_par.assign(c->n_gdn, 0);
        if (e == cudaSuccess) e = alloc_zero(&c->conv_w, (size_t)c->n_gdn * c->conv_ch * 4);
        if (e == cudaSuccess) e = alloc_zero(&c->conv_state, (size_t)2 * c->n_gdn * n_chars * 3 * c->conv_ch);
        if (e == cudaSuccess) e = alloc_zero(&c->conv_y, (size_t)max_tail_tokens * c->conv_ch);
    }
    if (c->n_attn) {
        const size_t rows = (size_t)kProbeMaxQueries * c->Hq;
        const size_t tiles = ((size_t)c->max_cap + kProbeKeys - 1) / kProbeKeys;
        if (e == cudaSuccess) e = alloc_zero(&c->probe_q, rows * c->D);
        if (e == cudaSuccess) e = alloc_zero(&c->probe_part, tiles * rows * 2);
        if (e == cudaSuccess) e = alloc_zero(&c->probe_rows, rows * 2);
    }
    const size_t part_slots = c->n_attn ? 2 * (size_t)attention_grid_cap(c->num_sms, c->D) : 0;
    if (e == cudaSuccess) e = alloc_zero(&c->part_o, part_slots * kAttnRows * c->D);
    if (e == cudaSuccess) e = alloc_zero(&c->part_ml, part_slots * kAttnRows * 2);
    if (e == cudaSuccess) e = alloc_zero(&c->tickets, (size_t)n_chars * (n_kv_slabs + 1));
    if (e == cudaSuccess) e = alloc_zero(&c->flags, n_flags * kFlagStride);
    if (e == cudaSuccess) e = alloc_zero(&c->err, 1);
    if (e == cudaSuccess) e = alloc_zero(&c->diag, 16);
    if (c->n_gdn > 0) {
        // one record per (64-token chunk, head); a character's tail adds at most one ragged chunk
        c->gdn_rec = gdn_record_bytes(c->dk, c->dv);
        const size_t chunks = (size_t)max_tail_tokens / 64 + n_chars;
        if (e == cudaSuccess) e = alloc_dev(c, &c->gdn_work, chunks * c->H * c->gdn_rec, "gdn_work", false);
        if (e == cudaSuccess) e = alloc_dev(c, &c->gdn_flags, chunks * c->H * 32, "gdn_flags");
        if (c->dk == 128 && c->dv == 128) {
            c->gdn_snap_bytes = gdn_snapshot_bytes(c->dk, c->dv);
            if (e == cudaSuccess) e = alloc_dev(c, &c->gdn_snap, chunks * c->H * c->gdn_snap_bytes, "gdn_snap", false);
        }
    }
    {
        size_t total_stage = 0;
        auto take = [&](size_t bytes) { const size_t off = total_stage; total_stage += (bytes + 255) / 256 * 256; return off; };
        const size_t T = (size_t)max_tail_tokens;
        for (int l = 0; l < c->n_layers; ++l) {
            const bool attn = c->kind[l] == KVM_LAYER_ATTN;
            c->stage_in_off.push_back(take(T * (attn ? c->Hq * c->D : c->H * c->dk) * 2));    // q
            c->stage_in_off.push_back(take(T * (attn ? c->Hkv * c->D : c->H * c->dk) * 2));   // k
            c->stage_in_off.push_back(take(T * (attn ? c->Hkv * c->D : c->H * c->dv) * 2));   // v
            c->stage_in_off.push_back(attn ? 0 : take(T * c->H * 4));                        // alpha
            c->stage_in_off.push_back(attn ? 0 : take(T * c->H * 4));                        // beta
            c->stage_out_off.push_back(take(T * (attn ? c->Hq * c->D : c->H * c->dv) * 2));  // out
        }
        if (e == cudaSuccess) e = alloc_dev(c, &c->stage, total_stage, "stage", false);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_start, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_copies, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&c->compact_stream, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_round, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_compacted, cudaEventDisableTiming);
        c->ev_piece_go.assign(c->n_attn, nullptr);
        c->ev_piece_done.assign(c->n_attn, nullptr);
        for (int a = 0; a < c->n_attn && e == cudaSuccess; ++a) {
            e = cudaEventCreateWithFlags(&c->ev_piece_go[a], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_piece_done[a], cudaEventDisableTiming);
        }
        c->ev_in.assign(c->n_layers, nullptr);
        c->ev_done.assign(c->n_layers, nullptr);
        for (int l = 0; l < c->n_layers && e == cudaSuccess; ++l) {
            e = cudaEventCreateWithFlags(&c->ev_in[l], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_done[l], cudaEventDisableTiming);
        }
    }
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        free_all(c);
        delete c;
        return fail(KVM_E_CUDA, "allocation failed: %s", cudaGetErrorString(e));
    }
    if (c->n_attn > 0) {
        // TMA maps: rotated q as [max_tail][Hq][D] with a (64, g, 128/g) box;
        // every layer's K and V as rows of D with a (64, 64) box
        const uint64_t row_bytes = (uint64_t)c->D * 2;
        const uint64_t kd[2] = {(uint64_t)c->D, (uint64_t)c->n_attn * c->Hkv * c->T_cap};
        const uint64_t ks[1] = {row_bytes};
        const uint32_t kb[2] = {64, 64};
        if (kd[1] > (uint64_t)INT32_MAX ||
            !encode_bf16_sw128(&c->tmap_k, c->K, 2, kd, ks, kb) ||
            !encode_bf16_sw128(&c->tmap_v, c->V, 2, kd, ks, kb)) {
            free_all(c);
            delete c;
            return fail(KVM_E_CUDA, "creating the TMA tensor maps failed");
        }
    }
    *out = c;
    return KVM_OK;
}

extern "C" kvm_status kvm_destroy(kvm_ctx* c) {
    if (!c) return KVM_OK;
    cudaDeviceSynchronize();
    free_all(c);
    delete c;
    return KVM_OK;
}

extern "C" const char* kvm_last_error(void) { return g_err.c_str(); }

extern "C" int64_t kvm_launch_count(const kvm_ctx* c) { return c ? c->launches : 0; }

// ============================================================================
// state access
// ============================================================================
extern "C" kvm_status kvm_load_prefix(kvm_ctx* c, int32_t b, int32_t live, int64_t cursor,
                                      const int32_t* positions, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    if (live < 0 || live > c->cap[b]) return fail(KVM_E_CAPACITY, "live %d exceeds capacity %d", live, c->cap[b]);
    if (live > 0 && !positions) return fail(KVM_E_INVAL, "positions is NULL");
    for (int i = 0; i < live; ++i) {
        if (positions[i] < 0 || (i > 0 && positions[i] <= positions[i - 1]))
            return fail(KVM_E_INVAL, "positions must be non-negative and strictly increasing");
    }
    if (live > 0 && cursor <= positions[live - 1]) return fail(KVM_E_INVAL, "cursor must exceed every position");
    if (cursor < 0 || cursor + c->max_tail > INT32_MAX) return fail(KVM_E_INVAL, "cursor out of range");
    cudaStream_t s = (cudaStream_t)stream;
    if (c->n_attn && live > 0) {
        CUDA_TRY(cudaMemcpyAsync(c->pos + c->cap_off[b], positions, (size_t)live * 4, cudaMemcpyHostToDevice, s));
        CUDA_TRY(cudaStreamSynchronize(s));
    }
    c->live[b] = live;
    c->cursor[b] = cursor;
    c->hpos[b].assign(positions, positions + live);
    return KVM_OK;
}

extern "C" kvm_status kvm_set_kv(kvm_ctx* c, int32_t layer, int32_t b, const void* k, const void* v,
                                 void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_layer(c, layer, KVM_LAYER_ATTN);
    if (st) return st;
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    const int L = c->live[b];
    if (L == 0) return KVM_OK;
    if (!k || !v) return fail(KVM_E_INVAL, "NULL k or v");
    const size_t row = (size_t)c->D * 2;
    const size_t slab = (size_t)c->T_cap * row;
    const int a = c->attn_idx[layer];
    char* kd = reinterpret_cast<char*>(c->K) + ((size_t)a * c->Hkv) * slab + (size_t)c->cap_off[b] * row;
    char* vd = reinterpret_cast<char*>(c->V) + ((size_t)a * c->Hkv) * slab + (size_t)c->cap_off[b] * row;
    cudaStream_t s = (cudaStream_t)stream;
    CUDA_TRY(cudaMemcpy2DAsync(kd, slab, k, L * row, L * row, c->Hkv, cudaMemcpyDeviceToDevice, s));
    CUDA_TRY(cudaMemcpy2DAsync(vd, slab, v, L * row, L * row, c->Hkv, cudaMemcpyDeviceToDevice, s));
    return KVM_OK;
}

extern "C" kvm_status kvm_get_kv(kvm_ctx* c, int32_t layer, int32_t b, void* k, void* v, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_layer(c, layer, KVM_LAYER_ATTN);
    if (st) return st;
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    const int L = c->live[b];
    if (L == 0) return KVM_OK;
    if (!k || !v) return fail(KVM_E_INVAL, "NULL k or v");
    const size_t row = (size_t)c->D * 2;
    const size_t slab = (size_t)c->T_cap * row;
    const int a = c->attn_idx[layer];
    const char* ks = reinterpret_cast<const char*>(c->K) + ((size_t)a * c->Hkv) * slab + (size_t)c->cap_off[b] * row;
    const char* vs = reinterpret_cast<const char*>(c->V) + ((size_t)a * c->Hkv) * slab + (size_t)c->cap_off[b] * row;
    cudaStream_t s = (cudaStream_t)stream;
    CUDA_TRY(cudaMemcpy2DAsync(k, L * row, ks, slab, L * row, c->Hkv, cudaMemcpyDeviceToDevice, s));
    CUDA_TRY(cudaMemcpy2DAsync(v, L * row, vs, slab, L * row, c->Hkv, cudaMemcpyDeviceToDevice, s));
    return KVM_OK;
}

extern "C" kvm_status kvm_get_positions(kvm_ctx* c, int32_t b, int32_t* out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    if (c->live[b] == 0 || c->n_attn == 0) return KVM_OK;
    if (!out) return fail(KVM_E_INVAL, "NULL output");
    CUDA_TRY(cudaMemcpyAsync(out, c->pos + c->cap_off[b], (size_t)c->live[b] * 4, cudaMemcpyDeviceToDevice,
                             (cudaStream_t)stream));
    return KVM_OK;
}

extern "C" kvm_status kvm_set_state(kvm_ctx* c, int32_t layer, const float* S, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_layer(c, layer, KVM_LAYER_GDN);
    if (st) return st;
    if (!S) return fail(KVM_E_INVAL, "NULL state");
    const size_t n = (size_t)c->B * c->H * c->dv * c->dk;
    CUDA_TRY(cudaMemcpyAsync(c->S + (size_t)c->gdn_idx[layer] * n, S, n * 4, cudaMemcpyDeviceToDevice,
                             (cudaStream_t)stream));
    return KVM_OK;
}

extern "C" kvm_status kvm_get_state(kvm_ctx* c, int32_t layer, float* S, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_layer(c, layer, KVM_LAYER_GDN);
    if (st) return st;
    if (!S) return fail(KVM_E_INVAL, "NULL state");
    const size_t n = (size_t)c->B * c->H * c->dv * c->dk;
    CUDA_TRY(cudaMemcpyAsync(S, c->S + (size_t)c->gdn_idx[layer] * n, n * 4, cudaMemcpyDeviceToDevice,
                             (cudaStream_t)stream));
    return KVM_OK;
}

namespace {
kvm_status check_conv_layer(const kvm_ctx* c, int layer) {
    kvm_status st = check_layer(c, layer, KVM_LAYER_GDN);
    if (st) return st;
    if (!c->conv) return fail(KVM_E_INVAL, "the context has no short convolution (conv_kernel = 0)");
    return KVM_OK;
}
// Current conv state buffer of a delta-rule layer ([B][3][C] bf16).
__nv_bfloat16* conv_state_of(kvm_ctx* c, int g, int which) {
    return c->conv_state + ((size_t)which * c->n_gdn + g) * c->B * 3 * c->conv_ch;
}
}  // namespace

extern "C" kvm_status kvm_set_conv_weights(kvm_ctx* c, int32_t layer, const float* w, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_conv_layer(c, layer);
    if (st) return st;
    if (!w) return fail(KVM_E_INVAL, "NULL weights");
    const size_t n = (size_t)c->conv_ch * 4;
    CUDA_TRY(cudaMemcpyAsync(c->conv_w + (size_t)c->gdn_idx[layer] * n, w, n * 4, cudaMemcpyDeviceToDevice,
                             (cudaStream_t)stream));
    return KVM_OK;
}

extern "C" kvm_status kvm_get_conv_state(kvm_ctx* c, int32_t layer, void* out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_conv_layer(c, layer);
    if (st) return st;
    if (!out) return fail(KVM_E_INVAL, "NULL output");
    const int g = c->gdn_idx[layer];
    CUDA_TRY(cudaMemcpyAsync(out, conv_state_of(c, g, c->conv_par[g]), (size_t)c->B * 3 * c->conv_ch * 2,
                             cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
    return KVM_OK;
}

extern "C" kvm_status kvm_set_conv_state(kvm_ctx* c, int32_t layer, const void* in, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_conv_layer(c, layer);
    if (st) return st;
    if (!in) return fail(KVM_E_INVAL, "NULL state");
    const int g = c->gdn_idx[layer];
    CUDA_TRY(cudaMemcpyAsync(conv_state_of(c, g, c->conv_par[g]), in, (size_t)c->B * 3 * c->conv_ch * 2,
                             cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
    return KVM_OK;
}

extern "C" kvm_status kvm_get_live(kvm_ctx* c, int32_t b, int32_t* live, int64_t* cursor) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    if (live) *live = c->live[b];
    if (cursor) *cursor = c->cursor[b];
    return KVM_OK;
}

// ============================================================================
// host-only planning (no context, no device)
// ============================================================================
extern "C" kvm_status kvm_plan_removal(int32_t n_chars, const int32_t* live, const int32_t* span_cu,
                                       const int32_t* span_begin, const int32_t* span_end, int32_t* new_live,
                                       int32_t* first_moved) {
    if (n_chars <= 0 || n_chars > kMaxChars) return fail(KVM_E_INVAL, "n_chars must be in [1,%d]", kMaxChars);
    if (!live) return fail(KVM_E_INVAL, "live is NULL");
    std::vector<int> L(live, live + n_chars);
    for (int b = 0; b < n_chars; ++b)
        if (L[b] < 0) return fail(KVM_E_INVAL, "negative live length at character %d", b);
    SpanPlan pl;
    const kvm_status st = plan_spans_for(n_chars, L.data(), span_cu, span_begin, span_end, pl);
    if (st) return st;
    for (int b = 0; b < n_chars; ++b) {
        if (new_live) new_live[b] = pl.L_new[b];
        if (first_moved) first_moved[b] = pl.first[b];
    }
    return KVM_OK;
}

extern "C" kvm_status kvm_plan_attention(int32_t n_chars, const int32_t* live, const int32_t* tail_cu,
                                         int32_t n_q_heads, int32_t n_kv_heads, int32_t max_blocks,
                                         int32_t* n_blocks, int32_t* n_tiles, int32_t* block_tile,
                                         int32_t* block_key, int32_t* n_split, int32_t* split_first_block) {
    if (n_chars <= 0 || n_chars > kMaxChars) return fail(KVM_E_INVAL, "n_chars must be in [1,%d]", kMaxChars);
    if (!live || !tail_cu || !n_blocks || !n_tiles || !block_tile || !block_key || !n_split || !split_first_block)
        return fail(KVM_E_INVAL, "NULL argument");
    if (n_kv_heads <= 0 || n_q_heads <= 0 || n_q_heads % n_kv_heads)
        return fail(KVM_E_UNSUPPORTED, "n_q_heads must be a multiple of n_kv_heads");
    const int g = n_q_heads / n_kv_heads;
    if (g > 64 || (g & (g - 1))) return fail(KVM_E_UNSUPPORTED, "group size must be a power of two <= 64");
    if (max_blocks <= 0 || max_blocks > kMaxAttnCtas)
        return fail(KVM_E_INVAL, "max_blocks must be in [1,%d]", kMaxAttnCtas);
    if (tail_cu[0] != 0) return fail(KVM_E_INVAL, "tail_cu[0] must be 0");
    std::vector<int> L(live, live + n_chars), M(n_chars);
    for (int b = 0; b < n_chars; ++b) {
        M[b] = tail_cu[b + 1] - tail_cu[b];
        if (M[b] < 0) return fail(KVM_E_INVAL, "tail_cu not monotone at character %d", b);
        if (L[b] < 0) return fail(KVM_E_INVAL, "negative live length at character %d", b);
    }
    AttnPlan pl;
    plan_attention(n_chars, L.data(), M.data(), n_kv_heads, kAttnRows / g, max_blocks, pl);
    *n_blocks = pl.n_ctas;
    *n_tiles = pl.n_tiles;
    std::copy(pl.cta_tile.begin(), pl.cta_tile.end(), block_tile);
    std::copy(pl.cta_k.begin(), pl.cta_k.end(), block_key);
    *n_split = (int32_t)pl.split_cb.size();
    std::copy(pl.split_cb.begin(), pl.split_cb.end(), split_first_block);
    return KVM_OK;
}

extern "C" kvm_status kvm_plan_partition(int32_t n_chars, const int64_t* cost, int32_t n_ranks, int32_t* rank_of,
                                         int64_t* rank_cost) {
    if (n_chars < 0 || n_ranks < 1) return fail(KVM_E_INVAL, "need n_chars >= 0 and n_ranks >= 1");
    if (n_chars > 0 && (!cost || !rank_of)) return fail(KVM_E_INVAL, "NULL argument");
    for (int b = 0; b < n_chars; ++b)
        if (cost[b] < 0) return fail(KVM_E_INVAL, "cost of character %d is negative", b);
    // longest processing time first: characters by decreasing cost (ties by
    // index), each to the rank with the least cost so far (ties: lowest rank)
    std::vector<int> order(n_chars);
    for (int b = 0; b < n_chars; ++b) order[b] = b;
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
    std::vector<int64_t> load(n_ranks, 0);
    for (int b : order) {
        int best = 0;
        for (int r = 1; r < n_ranks; ++r)
            if (load[r] < load[best]) best = r;
        rank_of[b] = best;
        load[best] += cost[b];
    }
    if (rank_cost) std::copy(load.begin(), load.end(), rank_cost);
    return KVM_OK;
}

namespace {
// Position ranges -> live-index spans over the live positions P[live].
// Positions are in live order; they increase unless per-token positions or
// re-rotation placed entries out of order.  Each range must cover at least
// one live entry, and the entries it covers must be one contiguous run of
// live indices (always true when the positions increase).
kvm_status spans_from_positions(const int32_t* P, int live, int32_t n, const int64_t* pb, const int64_t* pe,
                                int32_t* sb, int32_t* se) {
    if (n < 0) return fail(KVM_E_INVAL, "negative count");
    if (n > 0 && (!pb || !pe || !sb || !se)) return fail(KVM_E_INVAL, "NULL argument");
    bool increasing = true;
    for (int i = 1; i < live && increasing; ++i) increasing = P[i] > P[i - 1];
    int64_t prev_end = INT64_MIN;
    for (int i = 0; i < n; ++i) {
        if (pb[i] >= pe[i]) return fail(KVM_E_SPAN, "position range %d is empty", i);
        if (pb[i] < prev_end) return fail(KVM_E_SPAN, "position range %d overlaps or precedes the previous one", i);
        prev_end = pe[i];
        int lo, hi;
        if (increasing) {
            lo = (int)(std::lower_bound(P, P + live, pb[i]) - P);
            hi = (int)(std::lower_bound(P, P + live, pe[i]) - P);
        } else {
            lo = live;
            hi = -1;
            int count = 0;
            for (int j = 0; j < live; ++j)
                if (P[j] >= pb[i] && P[j] < pe[i]) {
                    lo = std::min(lo, j);
                    hi = std::max(hi, j + 1);
                    ++count;
                }
            if (count > 0 && count != hi - lo)
                return fail(KVM_E_SPAN, "position range %d covers live entries that are not one contiguous run", i);
        }
        if (hi <= lo) return fail(KVM_E_SPAN, "position range %d covers no live entry", i);
        sb[i] = lo;
        se[i] = hi;
    }
    return KVM_OK;
}
}  // namespace

extern "C" kvm_status kvm_spans_from_positions(kvm_ctx* c, int32_t b, int32_t n, const int64_t* pb,
                                               const int64_t* pe, int32_t* sb, int32_t* se) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    const std::vector<int32_t>& P = c->hpos[b];
    return spans_from_positions(P.data(), (int)P.size(), n, pb, pe, sb, se);
}

extern "C" kvm_status kvm_plan_spans_from_positions(int32_t live, const int32_t* positions, int32_t n,
                                                    const int64_t* pos_begin, const int64_t* pos_end,
                                                    int32_t* span_begin, int32_t* span_end) {
    if (live < 0) return fail(KVM_E_INVAL, "negative live length");
    if (live > 0 && !positions) return fail(KVM_E_INVAL, "positions is NULL");
    for (int i = 0; i < live; ++i)
        if (positions[i] < 0) return fail(KVM_E_INVAL, "positions must be non-negative");
    return spans_from_positions(positions, live, n, pos_begin, pos_end, span_begin, span_end);
}

// ============================================================================
// hot path
// ============================================================================
namespace {

// Compaction of the attention layers [a_lo, a_hi) (K and V slabs of those
// layers, and the position slab when with_pos) under a validated plan.
kvm_status launch_compaction(kvm_ctx* c, const SpanPlan& pl, cudaStream_t s, int a_lo, int a_hi, bool with_pos) {
    if (c->n_attn > 0 && a_hi > a_lo) {
        thread_local static CompactParams p;   // large parameter block, copied into the launch
        std::memset(&p, 0, sizeof p);
        p.n_chars = c->B;
        p.n_kv_slabs = 2 * (a_hi - a_lo) * c->Hkv;
        p.vec_per_row = c->D * 2 / 16;
        p.rows_kv = c->rows_kv;
        p.rows_pos = c->rows_pos;
        p.epoch = ++c->epoch;
        p.slab_rows = c->T_cap;
        p.K = reinterpret_cast<uint4*>(c->K + (size_t)a_lo * c->Hkv * c->T_cap * c->D);
        p.V = reinterpret_cast<uint4*>(c->V + (size_t)a_lo * c->Hkv * c->T_cap * c->D);
        p.pos = c->pos;
        p.tickets = c->tickets;
        p.flags = c->flags;
        p.flag_stride = kFlagStride;
        p.err = c->err;
        p.wait_limit = c->compact_wait_limit;
        // diag[15] is never written by any kernel (kvm_check clears it to 0,
        // and epochs start at 1), so a wait on it can only expire
        p.never_set = c->compact_stall ? reinterpret_cast<const uint32_t*>(c->diag + 15) : nullptr;
        int blk = 0;
        for (int b = 0; b < c->B; ++b) {
            CompactChar& ch = p.ch[b];
            const int moved = pl.n_seg[b] > 0 ? pl.L_new[b] - pl.first[b] : 0;
            ch.L_new = pl.L_new[b];
            ch.first = pl.first[b];
            ch.seg_off = pl.seg_off[b];
            ch.n_seg = pl.n_seg[b];
            ch.cap_off = c->cap_off[b];
            ch.chunks_kv = (moved + p.rows_kv - 1) / p.rows_kv;
            ch.chunks_pos = with_pos ? (moved + p.rows_pos - 1) / p.rows_pos : 0;
            ch.blk_off = blk;
            ch.flag_off = c->flag_off[b];
            blk += p.n_kv_slabs * ch.chunks_kv + ch.chunks_pos;
        }
        p.total_blocks = blk;
        std::copy(pl.seg_start.begin(), pl.seg_start.end(), p.seg_start);
        std::copy(pl.seg_shift.begin(), pl.seg_shift.end(), p.seg_shift);
        if (blk > 0) {
            const int ps = prof_begin(c, KVM_K_COMPACT, s);
            launch_kv_compact(p, s);
            prof_end(c, ps, s);
            LAUNCH_CHECK(c);
        }
    }
    return KVM_OK;
}

// The optional gather map (new slot -> old slot) of a validated plan.
kvm_status launch_gather(kvm_ctx* c, const SpanPlan& pl, int32_t* gather_out, cudaStream_t s) {
    if (gather_out) {
        thread_local static GatherParams gp;
        std::memset(&gp, 0, sizeof gp);
        gp.n_chars = c->B;
        int tot = 0;
        for (int b = 0; b < c->B; ++b) {
            gp.out_off[b] = tot;
            gp.first[b] = pl.first[b];
            gp.seg_off[b] = pl.seg_off[b];
            gp.n_seg[b] = pl.n_seg[b];
            tot += pl.L_new[b];
        }
        gp.out_off[c->B] = tot;
        gp.total = tot;
        gp.out = gather_out;
        std::copy(pl.seg_start.begin(), pl.seg_start.end(), gp.seg_start);
        std::copy(pl.seg_shift.begin(), pl.seg_shift.end(), gp.seg_shift);
        if (tot > 0) {
            const int ps = prof_begin(c, KVM_K_GATHER, s);
            launch_gather_map(gp, s);
            prof_end(c, ps, s);
            LAUNCH_CHECK(c);
        }
    }
    return KVM_OK;
}

// Host bookkeeping of a validated plan: live lengths and the position mirror.
void apply_plan(kvm_ctx* c, const SpanPlan& pl, const int32_t* span_cu, const int32_t* sbeg, const int32_t* send) {
    // host bookkeeping: live lengths and the position mirror
    for (int b = 0; b < c->B; ++b) {
        if (pl.n_seg[b] == 0) continue;
        std::vector<int32_t>& P = c->hpos[b];
        std::vector<int32_t> keep;
        keep.reserve(pl.L_new[b]);
        int k = span_cu[b];
        for (int i = 0; i < (int)P.size(); ++i) {
            while (k < span_cu[b + 1] && i >= send[k]) ++k;
            if (k < span_cu[b + 1] && i >= sbeg[k]) continue;
            keep.push_back(P[i]);
        }
        P.swap(keep);
        c->live[b] = pl.L_new[b];
    }
}


kvm_status do_compact(kvm_ctx* c, const int32_t* span_cu, const int32_t* sbeg, const int32_t* send,
                      int32_t* gather_out, cudaStream_t s) {
    SpanPlan pl;
    kvm_status st = plan_spans(c, span_cu, sbeg, send, pl);
    if (st) return st;
    st = launch_compaction(c, pl, s, 0, c->n_attn, true);
    if (st) return st;
    st = launch_gather(c, pl, gather_out, s);
    if (st) return st;
    apply_plan(c, pl, span_cu, sbeg, send);
    return KVM_OK;
}

// tail_pos_dev: device positions of the tail tokens (already staged), or
// null for the true tail p_b + i; tail_pos_host: the same values on the host
// for validation (null when tail_pos_dev is null).
kvm_status do_attention(kvm_ctx* c, int layer, const int32_t* tail_cu, const void* q, const void* k_new,
                        const void* v_new, void* out, cudaStream_t s, const int32_t* tail_pos_dev = nullptr,
                        const int32_t* tail_pos_host = nullptr) {
    kvm_status st = check_layer(c, layer, KVM_LAYER_ATTN);
    if (st) return st;
    int total = 0;
    st = check_tail_cu(c, tail_cu, &total);
    if (st) return st;
    for (int b = 0; b < c->B; ++b) {
        const int m = tail_cu[b + 1] - tail_cu[b];
        if (c->live[b] + m > c->cap[b])
            return fail(KVM_E_CAPACITY, "character %d: live %d + tail %d exceeds capacity %d", b, c->live[b], m,
                        c->cap[b]);
    }
    st = check_positions(c, tail_cu, tail_pos_host);
    if (st) return st;
    if (total == 0) return KVM_OK;
    if (!q || !k_new || !v_new || !out) return fail(KVM_E_INVAL, "NULL tensor");

    thread_local static AttnParams p;
    std::memset(&p, 0, sizeof p);
    const int a = c->attn_idx[layer];
    p.tmap_k = c->tmap_k;
    p.tmap_v = c->tmap_v;
    p.attn_layer = a;
    p.n_chars = c->B;
    p.Hq = c->Hq; p.Hkv = c->Hkv; p.D = c->D; p.R = c->R; p.g = c->g;
    p.tok_per_tile = kAttnRows / c->g;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c->D));
    p.slab_rows = c->T_cap;
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.k_new = static_cast<const __nv_bfloat16*>(k_new);
    p.v_new = static_cast<const __nv_bfloat16*>(v_new);
    p.q_rot = c->q_rot;
    p.K = c->K + (size_t)a * c->Hkv * c->T_cap * c->D;
    p.V = c->V + (size_t)a * c->Hkv * c->T_cap * c->D;
    p.pos = c->pos;
    p.out = static_cast<__nv_bfloat16*>(out);
    p.tail_pos = tail_pos_dev;
    p.part_o = c->part_o;
    p.part_ml = c->part_ml;
    p.err = c->err;
    p.diag = c->diag;
    for (int d = 0; d < c->R / 2; ++d) p.inv_freq[d] = c->inv_freq[d];
    std::vector<int> Ms(c->B);
    for (int b = 0; b < c->B; ++b) {
        AttnChar& ch = p.ch[b];
        ch.L_prev = c->live[b];
        ch.M = Ms[b] = tail_cu[b + 1] - tail_cu[b];
        ch.tail_off = tail_cu[b];
        ch.cap_off = c->cap_off[b];
        ch.p = c->cursor[b];
    }
    AttnPlan pl;
    plan_attention(c->B, c->live.data(), Ms.data(), c->Hkv, p.tok_per_tile, attention_grid_cap(c->num_sms, c->D), pl);
    for (int b = 0; b < c->B; ++b) {
        p.ch[b].n_qtiles = pl.n_qtiles[b];
        p.ch[b].tile_off = pl.tile_off[b];
    }
    p.n_tiles = pl.n_tiles;
    p.n_ctas = pl.n_ctas;
    std::copy(pl.cta_tile.begin(), pl.cta_tile.end(), p.cta_tile);
    std::copy(pl.cta_k.begin(), pl.cta_k.end(), p.cta_k);
    p.n_split_tiles = (int)pl.split_cb.size();
    std::copy(pl.split_cb.begin(), pl.split_cb.end(), p.split_cb);
    const bool split_tiles = p.n_split_tiles > 0;

    int ps = prof_begin(c, KVM_K_ROPE_APPEND, s);
    launch_rope_append(p, total, s);
    prof_end(c, ps, s);
    LAUNCH_CHECK(c);
    ps = prof_begin(c, KVM_K_ATTENTION, s);
    launch_tail_attention(p, s);
    prof_end(c, ps, s);
    LAUNCH_CHECK(c);
    if (split_tiles) {
        ps = prof_begin(c, KVM_K_ATTN_COMBINE, s);
        launch_attn_combine(p, s);
        prof_end(c, ps, s);
        LAUNCH_CHECK(c);
    }
    return KVM_OK;
}

kvm_status do_gdn(kvm_ctx* c, int layer, const int32_t* tail_cu, const void* q, const void* k, const void* v,
                  const float* alpha, const float* beta, void* out, cudaStream_t s) {
    kvm_status st = check_layer(c, layer, KVM_LAYER_GDN);
    if (st) return st;
    int total = 0;
    st = check_tail_cu(c, tail_cu, &total);
    if (st) return st;
    if (total == 0) return KVM_OK;
    if (!q || !k || !v || !alpha || !beta || !out) return fail(KVM_E_INVAL, "NULL tensor");
    thread_local static GdnParams p;
    std::memset(&p, 0, sizeof p);
    p.n_chars = c->B;
    p.H = c->H; p.dk = c->dk; p.dv = c->dv;
    // d_v rows of a head's state per scan block: split the rows (down to 32)
    // until the (character, head, slice) blocks cover the SMs
    {
        int active = 0;
        for (int b = 0; b < c->B; ++b) active += (tail_cu[b + 1] > tail_cu[b]);
        int slices = 1;
        while (c->dv / (2 * slices) >= 32 && c->dv % (2 * slices * 32) == 0 &&
               (int64_t)active * c->H * slices < c->num_sms)
            slices *= 2;
        p.dv_slice = c->dv / slices;
    }
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.k = static_cast<const __nv_bfloat16*>(k);
    p.v = static_cast<const __nv_bfloat16*>(v);
    if (c->conv) {
        // short convolution + SiLU (+ k normalisation) from the carried conv
        // state; the delta rule then reads the convolved q, k, v
        thread_local static ConvParams cp;
        std::memset(&cp, 0, sizeof cp);
        const int g = c->gdn_idx[layer];
        cp.n_chars = c->B;
        cp.H = c->H; cp.dk = c->dk; cp.dv = c->dv; cp.channels = c->conv_ch;
        cp.total = total;
        for (int b = 0; b <= c->B; ++b) cp.tail_cu[b] = tail_cu[b];
        cp.xq = p.q; cp.xk = p.k; cp.xv = p.v;
        cp.w = c->conv_w + (size_t)g * c->conv_ch * 4;
        cp.state_in = conv_state_of(c, g, c->conv_par[g]);
        cp.state_out = conv_state_of(c, g, c->conv_par[g] ^ 1);
        cp.yq = c->conv_y;
        cp.yk = cp.yq + (size_t)total * c->H * c->dk;
        cp.yv = cp.yk + (size_t)total * c->H * c->dk;
        cp.err = c->err;
        const int ps = prof_begin(c, KVM_K_GDN_CONV, s);
        launch_gdn_conv(cp, s);
        prof_end(c, ps, s);
        LAUNCH_CHECK(c);
        c->conv_par[g] ^= 1;
        p.q = cp.yq; p.k = cp.yk; p.v = cp.yv;
    }
    p.alpha = alpha;
    p.beta = beta;
    p.out = static_cast<__nv_bfloat16*>(out);
    p.S = c->S + (size_t)c->gdn_idx[layer] * c->B * c->H * c->dv * c->dk;
    p.err = c->err;
    p.diag = c->diag;
    p.work = c->gdn_work;
    p.rec_bytes = c->gdn_rec;
    int chunks = 0;
    for (int b = 0; b < c->B; ++b) {
        p.ch[b].M = tail_cu[b + 1] - tail_cu[b];
        p.ch[b].tail_off = tail_cu[b];
        p.ch[b].chunk_off = chunks;
        chunks += (p.ch[b].M + 63) / 64;
    }
    p.total_chunks = chunks;
    // two prep blocks per (chunk, head) when both fit on the SMs at once: they
    // share the solve for X and halve the products, staging and record
    // stores that follow it
    p.prep_parts = (int64_t)2 * chunks * c->H <= c->num_sms ? 2 : 1;
    // One launch for both when the scan items leave enough SMs to prep
    // workers (few characters) and the prep needs several rounds of them
    // (long tails): the chunk scan then starts on the first records while
    // the prep still works on later chunks.  Measured in a stack of
    // delta-rule layers (pipelined launches): 59.6 against 62.3 us a layer
    // for a 1024-token tail, but 27.0 against 22.4 us for 256 tokens, whose
    // prep is a single wave either way.  Otherwise the prep grid, then the scan.
    const int items = c->B * c->H * (c->dv / p.dv_slice);
    const int workers = c->num_sms - items;
    const bool fuse = c->gdn_fuse && p.dv_slice <= 32 && workers >= kMinPrepWorkers && chunks * c->H >= 2 * workers;
    if (c->gdn_chain && c->gdn_snap && p.dv_slice == 32) {
        // state-chain form: the chain carries only S (one MMA batch a chunk),
        // the outputs follow in a parallel pass over per-chunk snapshots
        p.snap = c->gdn_snap;
        p.snap_bytes = c->gdn_snap_bytes;
        p.n_scan = items;
        p.flags = c->gdn_flags;
        if (fuse) p.epoch = ++c->gdn_epoch;
        const int ps = prof_begin(c, KVM_K_GDN, s);
        const cudaError_t e = launch_gdn_v2(p, fuse ? std::min(c->num_sms, items + chunks * c->H) : 0, s);
        prof_end(c, ps, s);
        if (e == cudaSuccess) {
            LAUNCH_CHECK(c);
            return KVM_OK;
        }
        (void)cudaGetLastError();                     // the fused launch was refused: two launches from now on
        c->gdn_fuse = false;
        const int ps2 = prof_begin(c, KVM_K_GDN, s);
        const cudaError_t e2 = launch_gdn_v2(p, 0, s);
        prof_end(c, ps2, s);
        if (e2 != cudaSuccess) return fail(KVM_E_CUDA, "delta-rule launch failed: %s", cudaGetErrorString(e2));
        LAUNCH_CHECK(c);
        return KVM_OK;
    }
    if (fuse) {
        p.n_scan = items;
        p.epoch = ++c->gdn_epoch;
        p.flags = c->gdn_flags;
        const int grid = std::min(c->num_sms, items + chunks * c->H);
        const int ps = prof_begin(c, KVM_K_GDN, s);
        const cudaError_t e = launch_gdn_fused(p, grid, s);
        prof_end(c, ps, s);
        if (e == cudaSuccess) return KVM_OK;
        (void)cudaGetLastError();                     // the launch was refused: use two launches from now on
        c->gdn_fuse = false;
    }
    int ps = prof_begin(c, KVM_K_GDN_PREP, s);
    launch_gdn_chunk_prep(p, s);
    prof_end(c, ps, s);
    LAUNCH_CHECK(c);
    ps = prof_begin(c, KVM_K_GDN, s);
    launch_gdn_chunk_scan(p, s);
    prof_end(c, ps, s);
    LAUNCH_CHECK(c);
    return KVM_OK;
}

// End of a round: live lengths grow by M; the host position mirror gets the
// tail's positions; the cursor moves to p + M (true tail) or, with per-token
// positions, past the largest position used (it never moves back).
void do_advance(kvm_ctx* c, const int32_t* tail_cu, const int32_t* tail_pos = nullptr) {
    for (int b = 0; b < c->B; ++b) {
        const int m = tail_cu[b + 1] - tail_cu[b];
        if (tail_pos) {
            int64_t top = c->cursor[b];
            for (int i = 0; i < m; ++i) {
                const int32_t x = tail_pos[tail_cu[b] + i];
                c->hpos[b].push_back(x);
                top = std::max<int64_t>(top, (int64_t)x + 1);
            }
            c->cursor[b] = top;
        } else {
            for (int i = 0; i < m; ++i) c->hpos[b].push_back((int32_t)(c->cursor[b] + i));
            c->cursor[b] += m;
        }
        c->live[b] += m;
    }
}

}  // namespace

extern "C" kvm_status kvm_kv_compact(kvm_ctx* c, const int32_t* span_cu, const int32_t* sb, const int32_t* se,
                                     int32_t* gather_out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    return do_compact(c, span_cu, sb, se, gather_out, (cudaStream_t)stream);
}

extern "C" kvm_status kvm_tail_attn_prefill(kvm_ctx* c, int32_t layer, const int32_t* tail_cu, const void* q,
                                            const void* k_new, const void* v_new, void* out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    return do_attention(c, layer, tail_cu, q, k_new, v_new, out, (cudaStream_t)stream);
}

extern "C" kvm_status kvm_tail_attn_prefill_at(kvm_ctx* c, int32_t layer, const int32_t* tail_cu,
                                               const int32_t* tail_pos, const void* q, const void* k_new,
                                               const void* v_new, void* out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (!tail_pos) return do_attention(c, layer, tail_cu, q, k_new, v_new, out, (cudaStream_t)stream);
    kvm_status st = check_layer(c, layer, KVM_LAYER_ATTN);
    if (st) return st;
    int total = 0;
    st = check_tail_cu(c, tail_cu, &total);
    if (st) return st;
    st = check_positions(c, tail_cu, tail_pos);
    if (st) return st;
    for (int b = 0; b < c->B; ++b)
        if (c->live[b] + tail_cu[b + 1] - tail_cu[b] > c->cap[b])
            return fail(KVM_E_CAPACITY, "character %d: live + tail exceeds capacity", b);
    if (total > 0 && (!q || !k_new || !v_new || !out)) return fail(KVM_E_INVAL, "NULL tensor");
    st = stage_positions(c, tail_pos, total, c->tail_pos_dev, (cudaStream_t)stream);
    if (st) return st;
    return do_attention(c, layer, tail_cu, q, k_new, v_new, out, (cudaStream_t)stream, c->tail_pos_dev, tail_pos);
}

extern "C" kvm_status kvm_rerotate_keys(kvm_ctx* c, int32_t b, int32_t live_begin, int32_t live_end,
                                        const int32_t* new_pos, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (c->n_attn == 0) return fail(KVM_E_INVAL, "the model has no attention layer");
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    if (!(0 <= live_begin && live_begin <= live_end && live_end <= c->live[b]))
        return fail(KVM_E_SPAN, "range [%d,%d) outside the live entries [0,%d)", live_begin, live_end, c->live[b]);
    const int n = live_end - live_begin;
    if (n == 0) return KVM_OK;
    if (!new_pos) return fail(KVM_E_INVAL, "new_pos is NULL");
    int64_t top = c->cursor[b];
    for (int i = 0; i < n; ++i) {
        if (new_pos[i] < 0) return fail(KVM_E_INVAL, "new position %d is negative", i);
        top = std::max<int64_t>(top, (int64_t)new_pos[i] + 1);
    }
    cudaStream_t s = (cudaStream_t)stream;
    kvm_status st = stage_positions(c, new_pos, n, c->reloc_pos_dev, s);
    if (st) return st;
    RerotateParams p;
    std::memset(&p, 0, sizeof p);
    p.n = n;
    p.n_attn = c->n_attn;
    p.Hkv = c->Hkv;
    p.D = c->D;
    p.R = c->R;
    p.slot0 = (int64_t)c->cap_off[b] + live_begin;
    p.slab_rows = c->T_cap;
    p.K = c->K;
    p.pos = c->pos;
    p.new_pos = c->reloc_pos_dev;
    p.err = c->err;
    for (int d = 0; d < c->R / 2; ++d) p.inv_freq[d] = c->inv_freq[d];
    ++c->launches;
    launch_rerotate(p, s);
    LAUNCH_CHECK(c);
    for (int i = 0; i < n; ++i) c->hpos[b][live_begin + i] = new_pos[i];
    c->cursor[b] = top;
    return KVM_OK;
}

extern "C" kvm_status kvm_attn_probe(kvm_ctx* c, int32_t layer, int32_t b, int32_t n_q, const void* q,
                                     float* probs_out, const int32_t* group_of, int32_t n_groups,
                                     float* group_mass_out, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    kvm_status st = check_layer(c, layer, KVM_LAYER_ATTN);
    if (st) return st;
    if (b < 0 || b >= c->B) return fail(KVM_E_INVAL, "character %d out of range", b);
    const int L = c->live[b];
    if (n_q < 1 || n_q > kProbeMaxQueries || n_q > L)
        return fail(KVM_E_INVAL, "n_q must be in [1, min(%d, live = %d)]", kProbeMaxQueries, L);
    if (!q || !probs_out) return fail(KVM_E_INVAL, "NULL q or probs_out");
    if (group_of && (n_groups < 1 || !group_mass_out))
        return fail(KVM_E_INVAL, "group_of needs n_groups >= 1 and group_mass_out");
    cudaStream_t s = (cudaStream_t)stream;
    ProbeParams p;
    std::memset(&p, 0, sizeof p);
    p.L = L;
    p.n_q = n_q;
    p.Hq = c->Hq; p.Hkv = c->Hkv; p.D = c->D; p.R = c->R; p.g = c->g;
    p.n_groups = group_of ? n_groups : 0;
    p.scale = (float)(1.0 / std::sqrt((double)c->D));
    p.slab_rows = c->T_cap;
    p.slot0 = c->cap_off[b];
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.q_rot = c->probe_q;
    p.K = c->K + (size_t)c->attn_idx[layer] * c->Hkv * c->T_cap * c->D;
    p.pos = c->pos;
    p.part = c->probe_part;
    p.row_ms = c->probe_rows;
    p.probs = probs_out;
    p.group_of = group_of;
    p.group_mass = group_mass_out;
    p.err = c->err;
    for (int d = 0; d < c->R / 2; ++d) p.inv_freq[d] = c->inv_freq[d];
    if (group_of) CUDA_TRY(cudaMemsetAsync(group_mass_out, 0, sizeof(float) * (size_t)n_groups, s));
    c->launches += 4;
    launch_attn_probe(p, s);
    LAUNCH_CHECK(c);
    return KVM_OK;
}

extern "C" kvm_status kvm_effective_group_count(int32_t n_groups, const double* mass, double* out) {
    if (n_groups < 1 || !mass || !out) return fail(KVM_E_INVAL, "need n_groups >= 1, mass and out");
    double tot = 0.0;
    for (int i = 0; i < n_groups; ++i) {
        if (!(mass[i] >= 0.0)) return fail(KVM_E_INVAL, "group mass %d is negative or NaN", i);
        tot += mass[i];
    }
    if (!(tot > 0.0)) return fail(KVM_E_INVAL, "the groups carry no mass");
    double h = 0.0;                                  // entropy of the normalised group probabilities
    for (int i = 0; i < n_groups; ++i) {
        const double a = mass[i] / tot;
        if (a > 0.0) h -= a * std::log(a);
    }
    *out = std::exp(h);
    return KVM_OK;
}

extern "C" kvm_status kvm_total_variation(int32_t n, const double* p, const double* q, double* out) {
    if (n < 0 || (n > 0 && (!p || !q)) || !out) return fail(KVM_E_INVAL, "need n >= 0, p, q and out");
    double d = 0.0;
    for (int i = 0; i < n; ++i) d += std::fabs(p[i] - q[i]);
    *out = 0.5 * d;
    return KVM_OK;
}

extern "C" kvm_status kvm_gdn_chunk_scan_from_state(kvm_ctx* c, int32_t layer, const int32_t* tail_cu,
                                                    const void* q, const void* k, const void* v,
                                                    const float* alpha, const float* beta, void* out,
                                                    void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    return do_gdn(c, layer, tail_cu, q, k, v, alpha, beta, out, (cudaStream_t)stream);
}

extern "C" kvm_status kvm_advance_at(kvm_ctx* c, const int32_t* tail_cu, const int32_t* tail_pos) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    int total = 0;
    kvm_status st = check_tail_cu(c, tail_cu, &total);
    if (st) return st;
    for (int b = 0; b < c->B; ++b)
        if (c->live[b] + tail_cu[b + 1] - tail_cu[b] > c->cap[b])
            return fail(KVM_E_CAPACITY, "character %d would exceed its capacity", b);
    st = check_positions(c, tail_cu, tail_pos);
    if (st) return st;
    do_advance(c, tail_cu, tail_pos);
    return KVM_OK;
}

extern "C" kvm_status kvm_advance(kvm_ctx* c, const int32_t* tail_cu) { return kvm_advance_at(c, tail_cu, nullptr); }

namespace {
// NVTX ranges (a tool such as Nsight Systems shows them; without one attached
// each push / pop is a few nanoseconds).  Popped on every return path.
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace

kvm_status update_round_impl(kvm_ctx* c, const kvm_round* r, void* stream);

extern "C" kvm_status kvm_update_round(kvm_ctx* c, const kvm_round* r, void* stream) {
    NvtxRange range("kvm_update_round");
    return update_round_impl(c, r, stream);
}

kvm_status update_round_impl(kvm_ctx* c, const kvm_round* r, void* stream) {
    if (!c || !r) return fail(KVM_E_INVAL, "NULL argument");
    cudaStream_t s = (cudaStream_t)stream;
    int total = 0;
    kvm_status st = check_tail_cu(c, r->tail_cu, &total);
    if (st) return st;
    if (!r->q || !r->k || !r->v || !r->out) return fail(KVM_E_INVAL, "NULL per-layer pointer array");
    // validate everything before the first launch: spans and capacity after removal
    {
        SpanPlan pl;
        st = plan_spans(c, r->span_cu, r->span_begin, r->span_end, pl);
        if (st) return st;
        for (int b = 0; b < c->B; ++b) {
            const int m = r->tail_cu[b + 1] - r->tail_cu[b];
            if (pl.L_new[b] + m > c->cap[b])
                return fail(KVM_E_CAPACITY, "character %d: live %d + tail %d exceeds capacity %d", b, pl.L_new[b],
                            m, c->cap[b]);
        }
        st = check_positions(c, r->tail_cu, r->tail_pos);
        if (st) return st;
        for (int l = 0; l < c->n_layers; ++l) {
            if (total > 0 && (!r->q[l] || !r->k[l] || !r->v[l] || !r->out[l]))
                return fail(KVM_E_INVAL, "layer %d has a NULL tensor", l);
            if (c->kind[l] == KVM_LAYER_GDN && total > 0 && (!r->alpha || !r->beta || !r->alpha[l] || !r->beta[l]))
                return fail(KVM_E_INVAL, "layer %d has NULL gates", l);
        }
    }
    // maintenance delimiters: tail-index spans [s, e) of each character's
    // tail, checked like removal spans against the tail length
    std::vector<int> tail_len(c->B);
    for (int b = 0; b < c->B; ++b) tail_len[b] = r->tail_cu[b + 1] - r->tail_cu[b];
    SpanPlan delim_plan;
    const bool has_delim = r->delim_cu && r->delim_cu[c->B] > 0;
    if (has_delim) {
        st = plan_spans_for(c->B, tail_len.data(), r->delim_cu, r->delim_begin, r->delim_end, delim_plan);
        if (st) return st;
    }
    const bool host_io = r->io_on_host && total > 0;
    auto sizes = [&](int l, size_t n[6]) {
        const bool attn = c->kind[l] == KVM_LAYER_ATTN;
        n[0] = (size_t)total * (attn ? c->Hq * c->D : c->H * c->dk) * 2;
        n[1] = (size_t)total * (attn ? c->Hkv * c->D : c->H * c->dk) * 2;
        n[2] = (size_t)total * (attn ? c->Hkv * c->D : c->H * c->dv) * 2;
        n[3] = n[4] = attn ? 0 : (size_t)total * c->H * 4;
        n[5] = (size_t)total * (attn ? c->Hq * c->D : c->H * c->dv) * 2;
    };
    // Host-resident rounds stage a layer's inputs q, k, v, alpha, beta back to
    // back from the layer's staging base (each piece rounded up to 16 bytes).
    // Pieces that also lie back to back in the caller's memory go up in one
    // copy: a copy costs ~5 us before its first byte, so a caller that keeps
    // a layer's inputs in one pinned arena pays that once per layer.
    auto stage_in = [&](int l, size_t off[5]) {
        size_t n[6];
        sizes(l, n);
        size_t o = c->stage_in_off[5 * l];
        for (int i = 0; i < 5; ++i) {
            off[i] = o;
            o += (n[i] + 15) / 16 * 16;
        }
    };
    if (host_io) {
        // every layer's inputs go up on the copy stream at once (after the work
        // already queued on s, which may still read the staging buffers)
        CUDA_TRY(cudaEventRecord(c->ev_start, s));
        CUDA_TRY(cudaStreamWaitEvent(c->copy_stream, c->ev_start, 0));
        for (int l = 0; l < c->n_layers; ++l) {
            size_t n[6], off[5];
            sizes(l, n);
            stage_in(l, off);
            const char* src[5] = {static_cast<const char*>(r->q[l]), static_cast<const char*>(r->k[l]),
                                  static_cast<const char*>(r->v[l]),
                                  r->alpha ? reinterpret_cast<const char*>(r->alpha[l]) : nullptr,
                                  r->beta ? reinterpret_cast<const char*>(r->beta[l]) : nullptr};
            for (int i = 0; i < 5;) {
                if (!n[i]) { ++i; continue; }
                // extend the run while the next piece follows in both places
                int j = i;
                size_t bytes = n[i];
                while (j + 1 < 5 && n[j + 1] && n[j] % 16 == 0 && src[j + 1] == src[j] + n[j]) {
                    ++j;
                    bytes += n[j];
                }
                CUDA_TRY(cudaMemcpyAsync(c->stage + off[i], src[i], bytes, cudaMemcpyHostToDevice, c->copy_stream));
                i = j + 1;
            }
            CUDA_TRY(cudaEventRecord(c->ev_in[l], c->copy_stream));
        }
    }
    // Compaction changes only the attention layers' caches.  When recurrent
    // layers come before the first attention layer, each attention layer's
    // cache is compacted on the compaction stream beside the recurrent layers
    // that precede it (after the attention layer before them has finished),
    // and s joins that piece at the attention layer; the positions go with
    // the first piece.  Otherwise one launch on s compacts every layer.
    int first_attn = c->n_layers;
    for (int l = c->n_layers - 1; l >= 0; --l)
        if (c->kind[l] == KVM_LAYER_ATTN) first_attn = l;
    const bool side = first_attn > 0 && first_attn < c->n_layers;
    SpanPlan pl;
    st = plan_spans(c, r->span_cu, r->span_begin, r->span_end, pl);
    if (st) return st;
    // piece a runs beside the layers from piece_at[a] up to its attention layer
    std::vector<int> piece_at(c->n_attn, 0);
    for (int l = 0, prev = -1; l < c->n_layers; ++l)
        if (c->kind[l] == KVM_LAYER_ATTN) {
            piece_at[c->attn_idx[l]] = prev + 1;
            prev = l;
        }
    std::vector<char> piece_out(c->n_attn, 0);       // launched and not yet joined
    auto launch_piece = [&](int a) -> kvm_status {
        NvtxRange range("kv_compact");
        CUDA_TRY(cudaEventRecord(c->ev_piece_go[a], s));
        CUDA_TRY(cudaStreamWaitEvent(c->compact_stream, c->ev_piece_go[a], 0));
        if (a == 0) {
            // the gather map depends on the plan only; the first piece's event covers it
            const kvm_status g = launch_gather(c, pl, r->gather_out, c->compact_stream);
            if (g) return g;
        }
        const kvm_status e = launch_compaction(c, pl, c->compact_stream, a, a + 1, a == 0);
        if (e) return e;
        CUDA_TRY(cudaEventRecord(c->ev_piece_done[a], c->compact_stream));
        piece_out[a] = 1;
        return KVM_OK;
    };
    auto join_piece = [&](int a) -> cudaError_t {
        if (!piece_out[a]) return cudaSuccess;
        piece_out[a] = 0;
        return cudaStreamWaitEvent(s, c->ev_piece_done[a], 0);
    };
    auto join = [&]() -> cudaError_t {                // every piece launched so far
        for (int a = 0; a < c->n_attn; ++a) {
            const cudaError_t e = join_piece(a);
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    };
    if (!side) {
        NvtxRange range("kv_compact");
        st = launch_gather(c, pl, r->gather_out, s);
        if (st) return st;
        st = launch_compaction(c, pl, s, 0, c->n_attn, true);
        if (st) return st;
    }
    apply_plan(c, pl, r->span_cu, r->span_begin, r->span_end);
    const bool with_pos = r->tail_pos && total > 0 && c->n_attn > 0;
    if (with_pos) {
        st = stage_positions(c, r->tail_pos, total, c->tail_pos_dev, s);
        if (st) return st;
    }
    for (int l = 0; l < c->n_layers; ++l) {
        const bool attn = c->kind[l] == KVM_LAYER_ATTN;
        if (side) {
            for (int a = 0; a < c->n_attn; ++a)
                if (piece_at[a] == l) {
                    st = launch_piece(a);
                    if (st) {
                        join();
                        return st;
                    }
                }
            if (attn) CUDA_TRY(join_piece(c->attn_idx[l]));
        }
        const void *q = r->q[l], *k = r->k[l], *v = r->v[l];
        const float *al = attn ? nullptr : r->alpha[l], *be = attn ? nullptr : r->beta[l];
        void* out = r->out[l];
        if (host_io) {
            CUDA_TRY(cudaStreamWaitEvent(s, c->ev_in[l], 0));
            size_t o[5];
            stage_in(l, o);
            q = c->stage + o[0]; k = c->stage + o[1]; v = c->stage + o[2];
            if (!attn) {
                al = reinterpret_cast<const float*>(c->stage + o[3]);
                be = reinterpret_cast<const float*>(c->stage + o[4]);
            }
            out = c->stage + c->stage_out_off[l];
        }
        {
            char name[48];
            snprintf(name, sizeof name, "layer %d (%s)", l, attn ? "attention" : "delta rule");
            NvtxRange range(name);
            st = attn ? do_attention(c, l, r->tail_cu, q, k, v, out, s, with_pos ? c->tail_pos_dev : nullptr,
                                     with_pos ? r->tail_pos : nullptr)
                      : do_gdn(c, l, r->tail_cu, q, k, v, al, be, out, s);
        }
        if (st) {
            join();                                   // s still covers the compaction
            return st;
        }
        if (host_io) {
            // the layer's output goes down while the next layers compute
            size_t n[6];
            sizes(l, n);
            CUDA_TRY(cudaEventRecord(c->ev_done[l], s));
            CUDA_TRY(cudaStreamWaitEvent(c->copy_stream, c->ev_done[l], 0));
            CUDA_TRY(cudaMemcpyAsync(r->out[l], c->stage + c->stage_out_off[l], n[5], cudaMemcpyDeviceToHost,
                                     c->copy_stream));
        }
    }
    if (host_io) {
        // work queued on s after this round also follows the copies
        CUDA_TRY(cudaEventRecord(c->ev_copies, c->copy_stream));
        CUDA_TRY(cudaStreamWaitEvent(s, c->ev_copies, 0));
    }
    std::vector<int> L_round(c->live);              // L'_b: where each tail was appended
    do_advance(c, r->tail_cu, r->tail_pos);
    if (has_delim) {
        // the delimiters' direct KV leave every attention layer; their
        // effect on the recurrent states and on later tail tokens stays
        std::vector<int32_t> cu(c->B + 1), sb, se;
        for (int b = 0; b < c->B; ++b) {
            cu[b] = (int32_t)sb.size();
            for (int k = r->delim_cu[b]; k < r->delim_cu[b + 1]; ++k) {
                sb.push_back(L_round[b] + r->delim_begin[k]);
                se.push_back(L_round[b] + r->delim_end[k]);
            }
        }
        cu[c->B] = (int32_t)sb.size();
        SpanPlan pl;
        st = plan_spans(c, cu.data(), sb.data(), se.data(), pl);
        if (st) return st;                            // cannot happen: checked against the tails above
        st = launch_compaction(c, pl, s, 0, c->n_attn, true);
        if (st) return st;
        apply_plan(c, pl, cu.data(), sb.data(), se.data());
    }
    return KVM_OK;
}

namespace {
// The canary bands of every buffer, read back (debug builds; a no-op otherwise).
kvm_status check_canaries(kvm_ctx* c) {
    if (!kCanary) return KVM_OK;
    std::vector<unsigned char> band(kCanary);
    for (const auto& a : c->allocs) {
        for (int side = 0; side < 2; ++side) {
            const char* src = static_cast<const char*>(a.base) + (side ? kCanary + a.bytes : 0);
            CUDA_TRY(cudaMemcpy(band.data(), src, kCanary, cudaMemcpyDeviceToHost));
            for (size_t i = 0; i < kCanary; ++i)
                if (band[i] != kCanaryByte)
                    return fail(KVM_E_DEVICE, "canary band %s buffer %s overwritten (byte %zu)",
                                side ? "after" : "before", a.name, i);
        }
    }
    return KVM_OK;
}
}  // namespace

extern "C" kvm_status kvm_debug_poke_canary(kvm_ctx* c) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (!kCanary) return fail(KVM_E_UNSUPPORTED, "canary bands exist only in builds with -DKVM_DEBUG");
    if (c->allocs.empty()) return fail(KVM_E_INVAL, "the context owns no device buffer");
    const auto& a = c->allocs.front();
    CUDA_TRY(cudaDeviceSynchronize());
    CUDA_TRY(cudaMemset(static_cast<char*>(a.base) + kCanary + a.bytes, 0, 1));   // first byte past the buffer
    return KVM_OK;
}

extern "C" kvm_status kvm_check(kvm_ctx* c, void* stream) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    CUDA_TRY(cudaStreamSynchronize((cudaStream_t)stream));
    {
        const kvm_status cs = check_canaries(c);
        if (cs) return cs;
    }
    int32_t e = 0;
    CUDA_TRY(cudaMemcpy(&e, c->err, 4, cudaMemcpyDeviceToHost));
    if (e) {
        int32_t d[3] = {0, 0, 0};
        CUDA_TRY(cudaMemcpy(d, c->diag, sizeof d, cudaMemcpyDeviceToHost));
        CUDA_TRY(cudaMemset(c->err, 0, 4));
        CUDA_TRY(cudaMemset(c->diag, 0, 16 * sizeof(int32_t)));
        CUDA_TRY(cudaMemset(c->tickets, 0, sizeof(int32_t) * (size_t)c->B * (2 * c->n_attn * c->Hkv + 1)));
        return fail(KVM_E_DEVICE, "device error word 0x%x (%s%s); first expired wait: block %d, tag 0x%x, parity %d",
                    e, (e & kErrBounds) ? "bounds " : "", (e & kErrWait) ? "wait-timeout" : "", d[0] - 1, d[1], d[2]);
    }
    return KVM_OK;
}

extern "C" kvm_status kvm_set_plan(kvm_ctx* c, int32_t what, int32_t enable) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    switch (what) {
        case KVM_PLAN_GDN_FUSED: c->gdn_fuse = enable != 0; break;
        case KVM_PLAN_GDN_STATE_CHAIN: c->gdn_chain = enable != 0; break;
        default: return fail(KVM_E_INVAL, "unknown plan option %d", what);
    }
    return KVM_OK;
}

extern "C" kvm_status kvm_debug_compact_wait(kvm_ctx* c, int32_t polls, int32_t stall) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (polls < 0) return fail(KVM_E_INVAL, "polls must be >= 0");
    c->compact_wait_limit = polls ? polls : kCompactWaitLimit;
    c->compact_stall = stall != 0;
    return KVM_OK;
}

extern "C" kvm_status kvm_fork(kvm_ctx* dst, const kvm_ctx* src, void* stream) {
    if (!dst || !src) return fail(KVM_E_INVAL, "NULL context");
    if (dst == src) return KVM_OK;
    if (dst->kind != src->kind || dst->Hq != src->Hq || dst->Hkv != src->Hkv || dst->D != src->D ||
        dst->R != src->R || dst->theta != src->theta || dst->H != src->H || dst->dk != src->dk ||
        dst->dv != src->dv || dst->B != src->B || dst->cap != src->cap || dst->conv != src->conv)
        return fail(KVM_E_INVAL, "contexts differ in model shape, population or capacity");
    cudaStream_t s = (cudaStream_t)stream;
    const size_t kv = (size_t)src->n_attn * src->Hkv * src->T_cap * src->D * sizeof(__nv_bfloat16);
    if (kv) {
        CUDA_TRY(cudaMemcpyAsync(dst->K, src->K, kv, cudaMemcpyDeviceToDevice, s));
        CUDA_TRY(cudaMemcpyAsync(dst->V, src->V, kv, cudaMemcpyDeviceToDevice, s));
        CUDA_TRY(cudaMemcpyAsync(dst->pos, src->pos, (size_t)src->T_cap * 4, cudaMemcpyDeviceToDevice, s));
    }
    const size_t sn = (size_t)src->n_gdn * src->B * src->H * src->dv * src->dk * sizeof(float);
    if (sn) CUDA_TRY(cudaMemcpyAsync(dst->S, src->S, sn, cudaMemcpyDeviceToDevice, s));
    if (src->conv) {
        const size_t cs = (size_t)2 * src->n_gdn * src->B * 3 * src->conv_ch * 2;
        CUDA_TRY(cudaMemcpyAsync(dst->conv_state, src->conv_state, cs, cudaMemcpyDeviceToDevice, s));
        CUDA_TRY(cudaMemcpyAsync(dst->conv_w, src->conv_w, (size_t)src->n_gdn * src->conv_ch * 4 * 4,
                                 cudaMemcpyDeviceToDevice, s));
        dst->conv_par = src->conv_par;
    }
    dst->live = src->live;
    dst->cursor = src->cursor;
    dst->hpos = src->hpos;
    return KVM_OK;
}

extern "C" kvm_status kvm_profile_enable(kvm_ctx* c, int32_t enable) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (enable && c->ev.empty()) {
        c->ev.resize(2 * kProfPool);
        for (auto& e : c->ev) CUDA_TRY(cudaEventCreate(&e));
    }
    c->prof = enable != 0;
    return KVM_OK;
}

extern "C" kvm_status kvm_profile_read(kvm_ctx* c, int32_t kernel, int64_t* launches, double* total_ms,
                                       int32_t reset) {
    if (!c) return fail(KVM_E_INVAL, "NULL context");
    if (kernel < 0 || kernel >= KVM_K_COUNT) return fail(KVM_E_INVAL, "kernel family %d out of range", kernel);
    CUDA_TRY(cudaDeviceSynchronize());
    double ms = 0.0;
    int64_t timed = 0;                     // launches that got a pair of events
    for (size_t i = 0; i < c->ev_kind.size(); ++i) {
        if (c->ev_kind[i] != kernel) continue;
        float t = 0.f;
        CUDA_TRY(cudaEventElapsedTime(&t, c->ev[2 * i], c->ev[2 * i + 1]));
        ms += t;
        ++timed;
    }
    if (launches) *launches = timed;
    if (total_ms) *total_ms = ms;
    if (reset) c->ev_kind.clear();
    return KVM_OK;
}

namespace kvm {
// Lets other translation units of the library report a failure through
// kvm_last_error().
kvm_status report_error(kvm_status code, const char* msg) { return fail(code, "%s", msg); }
}  // namespace kvm
