// Causal GQA attention of the true tail over the compacted cache (Eq. 3 for a
// full-attention layer), on the sm_100-family tensor cores.
//
// Query tiles have 128 rows = (tail token, query head of one GQA group) pairs,
// token-major, so each K/V tile serves all g heads of the group.  The work is
// the list of (query tile, 64-key tile) units; it is cut into contiguous
// ranges, one per persistent block (stream-K), balanced by a cost model that
// charges each unit 1 and each segment a block starts 8 more (the host
// planner bisects for the smallest per-block cost).  A block's range covers whole
// query tiles, whose outputs it normalises and stores directly, and at most
// one partial tile at each end, whose unnormalised accumulator goes to a
// workspace slot (2c for block c's first segment, 2c + 1 for its last) for
// attn_combine.
//
// Roles of a block (384 threads):
//   warps 0, 11 TMA producers: lane 0 of warp 0 streams the K tiles, lane 0
//               of warp 11 the V tiles of each segment's keys, each through a
//               three-stage ring (64 keys x D, 128-byte swizzle); separate
//               warps keep the two rings from waiting on each other;
//   warp 1      allocates TMEM and issues S_j = Q K_j^T (tcgen05.mma,
//               M 128, N 64, K D, Q read from TMEM) into two TMEM buffers;
//   warp 10     issues O += P_j V_j (M 128, N D, K 64) into the TMEM
//               accumulator.  Two issuers keep the S stream running ahead of
//               the softmax while the PV stream follows it.  Each issuer warp
//               runs its loop converged and one elected lane issues: a lone
//               lane in a divergent branch issued the same MMAs at ~1.6x the
//               cycles per instruction;
//   warps 2-9   softmax: each query row is shared by the two warps that see
//               its TMEM lane quarter (warp w reads lanes 32 (w mod 4) ..),
//               one per 32-key half of S_j.  They stage the segment's Q tile
//               in TMEM (the next segment's as soon as the last S of the
//               current one has landed), exchange row maxima through shared
//               memory and a pair barrier, keep an online softmax in base 2
//               with lazy rescaling (the reference max moves only when a
//               score exceeds it by more than 2^8; the O row is then rescaled
//               in TMEM, each half its half of the columns) and write P_j as
//               bf16 into one of two shared buffers in the MMA's swizzled
//               K-major layout, so that the softmax of tile j+1 does not wait
//               for PV_j.  At the end of a segment each half stores its half
//               of the O columns.
// Q lives in TMEM rather than shared memory: S_j then reads only K_j from
// shared memory, and the space goes to a third K and V stage.
// Every mbarrier wait is bounded in time.  On expiry the block raises an
// abort flag and records kErrWait: the producers and the MMA issuer stop
// issuing, the softmax warps run their loops to the end without waiting (so
// that their pair barriers stay matched), and every copy and MMA already
// issued completes before TMEM and shared memory are released.
#include "kvm_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvm {
namespace {

using namespace ptx;

constexpr int BM = 128;                       // query rows per tile
constexpr int BN = 64;                        // keys per K/V tile
constexpr int kSoftmaxThreads = 256;          // warps 2-9
constexpr int kThreads = 64 + kSoftmaxThreads + 64;   // + warp 10 (PV issuer), warp 11 (V producer)
constexpr int kPvWarp = 10;
constexpr int kVWarp = 11;

constexpr int STAGES = 3;                     // K and V ring depth

enum Bar { K_FULL = 0, K_EMPTY = 3, V_FULL = 6, V_EMPTY = 9, S_FULL = 12, S_EMPTY = 14, P_FULL = 16,
           PV_DONE = 18, Q_FULL = 20, O_FINAL = 21, O_EMPTY = 22, DRAIN_S = 23, DRAIN_PV = 24, N_BARS = 25 };

template <int D>
struct Cfg {
    static constexpr int NREG = D / 64;                    // 64-column (128-byte) regions
    static constexpr int HALF = D / 2;                     // O columns per softmax half
    static constexpr int KV_BYTES = BN * D * 2;
    static constexpr int P_BYTES = BM * BN * 2;
    static constexpr int OFF_K = 0;
    static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
    static constexpr int OFF_P = OFF_V + STAGES * KV_BYTES;
    static constexpr int OFF_BAR = OFF_P + 2 * P_BYTES;
    static constexpr int OFF_SLOT = OFF_BAR + N_BARS * 8;  // TMEM base address
    static constexpr int OFF_ABORT = OFF_SLOT + 4;
    static constexpr int OFF_X = (OFF_ABORT + 4 + 15) / 16 * 16;   // float [2][2][BM] row exchange
    static constexpr int USED = OFF_X + 2 * 2 * BM * 4;
    // head_dim 256 leaves no room to align the base up: a block without static
    // shared variables gets a 1024-aligned dynamic base (checked at run time)
    static constexpr int SLACK = (D == 256) ? 0 : 1024;
    static constexpr int SMEM = USED + SLACK;
    static constexpr uint32_t TMEM_S = 0;                  // two S buffers of BN columns
    static constexpr uint32_t TMEM_O = 2 * BN;             // D columns
    static constexpr uint32_t TMEM_Q = 2 * BN + D;         // D / 2 columns: Q as bf16 pairs
    static constexpr uint32_t TMEM_COLS = (TMEM_Q + D / 2 <= 256) ? 256 : 512;
};
static_assert(Cfg<256>::SMEM <= 232448, "shared memory of the head_dim 256 attention");
static_assert(Cfg<256>::TMEM_Q + 128 <= 512, "TMEM of the head_dim 256 attention");

struct Tile {
    int b, kvh, qt, nk, tok0, tok_end;
};

// Query tile t -> (character, KV head, tile within the head) and its number
// of 64-key tiles (every surviving entry plus the tail up to its last token).
__device__ __forceinline__ Tile decode_tile(const AttnParams& p, int t) {
    int lo = 0, hi = p.n_chars - 1;               // last b with tile_off <= t
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].tile_off <= t) lo = mid; else hi = mid - 1;
    }
    Tile r;
    r.b = lo;
    const AttnChar& c = p.ch[lo];
    const int local = t - c.tile_off;
    r.kvh = local / c.n_qtiles;
    r.qt = local % c.n_qtiles;
    r.tok0 = r.qt * p.tok_per_tile;
    r.tok_end = min(c.M, r.tok0 + p.tok_per_tile);
    r.nk = (c.L_prev + r.tok_end + BN - 1) / BN;
    return r;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) tail_attention_tc_kernel(const __grid_constant__ AttnParams p) {
    using C = Cfg<D>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    uint8_t* smem = smem_raw;
    if (C::SLACK) {
        smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    } else if (smem_u32(smem_raw) & 1023u) {
        if (threadIdx.x == 0) atomicOr(p.err, kErrBounds);
        return;                                    // uniform: before any barrier or TMEM use
    }
    const uint32_t sbase = smem_u32(smem);
    const uint32_t sK = sbase + C::OFF_K, sV = sbase + C::OFF_V, sP = sbase + C::OFF_P;
    auto bar = [&](int i) -> uint32_t { return sbase + C::OFF_BAR + 8u * i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_SLOT);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_ABORT);
    float* xch = reinterpret_cast<float*>(smem + C::OFF_X);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int cta = blockIdx.x;
    const int g = p.g;
    const int t_begin = p.cta_tile[cta], k_begin = p.cta_k[cta];
    const int t_end = p.cta_tile[cta + 1], k_end = p.cta_k[cta + 1];
    auto more = [&](int t, int k) { return t < t_end || (t == t_end && k < k_end); };
    // A barrier wait of a whole issuer warp: lane 0 polls, the warp takes its result.
    auto warp_wait = [&](uint32_t b, uint32_t parity, int tag) -> bool {
        int r = 1;
        if ((threadIdx.x & 31) == 0) r = mbar_wait(b, parity, abort_flag, p.err, kErrWait, p.diag, tag) ? 1 : 0;
        return __shfl_sync(0xffffffffu, r, 0) != 0;
    };

    if (tid == 0) {
        *abort_flag = 0;
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(bar(K_FULL + s), 1);
            mbar_init(bar(K_EMPTY + s), 1);
            mbar_init(bar(V_FULL + s), 1);
            mbar_init(bar(V_EMPTY + s), 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(bar(S_FULL + s), 1);
            mbar_init(bar(S_EMPTY + s), kSoftmaxThreads);
            mbar_init(bar(P_FULL + s), kSoftmaxThreads);
            mbar_init(bar(PV_DONE + s), 1);
        }
        mbar_init(bar(Q_FULL), kSoftmaxThreads);
        mbar_init(bar(O_FINAL), 1);
        mbar_init(bar(O_EMPTY), kSoftmaxThreads);
        mbar_init(bar(DRAIN_S), 1);
        mbar_init(bar(DRAIN_PV), 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // The kernel before this one (rope_append) writes the tail's keys and
    // values and the rotated q; the surviving rows [0, L') were written
    // earlier (by kv_compact, complete before rope_append began).  So the
    // producers stream survivor tiles at once and wait for the previous grid
    // only before a tile that reaches the tail; the softmax warps wait before
    // staging Q.  The issuers touch no global memory.
    grid_dependents_launch();

    // copies issued by a producer lane (for the drain after an abort)
    int last_load[STAGES] = {-1, -1, -1};

    if (warp == 0 || warp == kVWarp) {
        // ------------------------------------------------------------ producers: warp 0 K, warp 11 V
        if (lane == 0) {
            const bool is_k = warp == 0;
            const CUtensorMap* map = is_k ? &p.tmap_k : &p.tmap_v;
            const uint32_t ring = is_k ? sK : sV;
            const int full = is_k ? K_FULL : V_FULL, empty = is_k ? K_EMPTY : V_EMPTY;
            prefetch_tmap(map);
            bool ok = true, waited = false;
            int j = 0;
            for (int t = t_begin, k = k_begin; ok && more(t, k); ++t, k = 0) {
                const Tile T = decode_tile(p, t);
                const AttnChar& ch = p.ch[T.b];
                const int k1 = (t == t_end) ? k_end : T.nk;
                const int key_row0 = (p.attn_layer * p.Hkv + T.kvh) * (int)p.slab_rows + ch.cap_off;
                for (int kt = k; kt < k1; ++kt, ++j) {
                    if (!waited && (kt + 1) * BN > ch.L_prev) {    // the tile reaches the tail
                        grid_dependency_wait();
                        waited = true;
                    }
                    const int st = j % STAGES;
                    if (j >= STAGES)
                        ok = mbar_wait(bar(empty + st), (j / STAGES - 1) & 1, abort_flag, p.err, kErrWait, p.diag,
                                       (is_k ? 0x12 : 0x13) + 256 * j);
                    if (!ok) break;
                    mbar_arrive_expect_tx(bar(full + st), C::KV_BYTES);
                    for (int r = 0; r < C::NREG; ++r)
                        tma_load_2d(ring + st * C::KV_BYTES + r * (BN * 128), map, r * 64, key_row0 + kt * BN, bar(full + st));
                    last_load[st] = j;
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ S issuer
        // The whole warp runs the loop; lane 0 polls the barriers and an
        // elected lane (lane 0 again) issues, so the descriptors stay warp-uniform.
        const uint32_t id_qk = idesc_bf16_f32(BM, BN, false);
        const uint64_t k_desc0 = smem_desc_sw128(sK, 16, 1024);   // + (byte offset >> 4) per operand
        bool ok = true;
        int j = 0, seg = 0;
        for (int t = t_begin, k = k_begin; ok && more(t, k); ++t, k = 0, ++seg) {
            const Tile T = decode_tile(p, t);
            const int n = ((t == t_end) ? k_end : T.nk) - k;
            ok = warp_wait(bar(Q_FULL), seg & 1, 0x21 + 256 * seg);
            for (int i = 0; i < n && ok; ++i, ++j) {
                const int sb = j & 1, st = j % STAGES;
                ok = warp_wait(bar(K_FULL + st), (j / STAGES) & 1, 0x22 + 256 * j);
                if (ok && j >= 2) ok = warp_wait(bar(S_EMPTY + sb), ((j >> 1) - 1) & 1, 0x23 + 256 * j);
                if (!ok) break;
                tc_fence_after();
                const uint64_t kd = k_desc0 + (uint64_t)((st * C::KV_BYTES) >> 4);
                const uint32_t d = tmem + C::TMEM_S + sb * BN;
                if (elect_one()) {
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks)
                        mma_bf16_ts(d, tmem + C::TMEM_Q + ks * 8, kd + (uint64_t)((((ks >> 2) * (BN * 128)) + (ks & 3) * 32) >> 4),
                                    id_qk, ks > 0);
                    mma_commit(bar(S_FULL + sb));
                    mma_commit(bar(K_EMPTY + st));
                }
                __syncwarp();
            }
        }
        // every MMA issued by this warp completes before TMEM is released
        if (elect_one()) mma_commit(bar(DRAIN_S));
        __syncwarp();
        volatile int never = 0;
        if (lane == 0) mbar_wait(bar(DRAIN_S), 0, &never, p.err, kErrWait, nullptr, 0, 1000000000ull);
        __syncwarp();
    } else if (warp == kPvWarp) {
        // ------------------------------------------------------------ PV issuer (same warp discipline)
        const uint32_t id_pv = idesc_bf16_f32(BM, D, true);
        const uint64_t p_desc0 = smem_desc_sw128(sP, 16, 1024);
        const uint64_t v_desc0 = smem_desc_sw128(sV, BN * 128, 1024);
        bool ok = true;
        int j = 0, seg = 0;
        for (int t = t_begin, k = k_begin; ok && more(t, k); ++t, k = 0, ++seg) {
            const Tile T = decode_tile(p, t);
            const int n = ((t == t_end) ? k_end : T.nk) - k;
            for (int i = 0; i < n && ok; ++i, ++j) {
                const int pb = j & 1, st = j % STAGES;
                ok = warp_wait(bar(P_FULL + pb), (j >> 1) & 1, 0x24 + 256 * j);
                if (ok) ok = warp_wait(bar(V_FULL + st), (j / STAGES) & 1, 0x25 + 256 * j);
                // the previous segment's O has been read out before it is overwritten
                if (ok && i == 0 && seg > 0) ok = warp_wait(bar(O_EMPTY), (seg - 1) & 1, 0x26 + 256 * seg);
                if (!ok) break;
                tc_fence_after();
                const uint64_t pd = p_desc0 + (uint64_t)((pb * C::P_BYTES) >> 4);
                const uint64_t vd = v_desc0 + (uint64_t)((st * C::KV_BYTES) >> 4);
                if (elect_one()) {
#pragma unroll
                    for (int ks = 0; ks < BN / 16; ++ks)
                        mma_bf16(tmem + C::TMEM_O, pd + (uint64_t)((ks * 32) >> 4), vd + (uint64_t)((ks * 16 * 128) >> 4), id_pv,
                                 (i > 0 || ks > 0) ? 1u : 0u);
                    mma_commit(bar(PV_DONE + pb));
                    mma_commit(bar(V_EMPTY + st));
                }
                __syncwarp();
            }
            if (ok) {
                if (elect_one()) mma_commit(bar(O_FINAL));
                __syncwarp();
            }
        }
        if (elect_one()) mma_commit(bar(DRAIN_PV));
        __syncwarp();
        volatile int never = 0;
        if (lane == 0) mbar_wait(bar(DRAIN_PV), 0, &never, p.err, kErrWait, nullptr, 0, 1000000000ull);
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int half = (warp - 2) >> 2;                  // key columns 32 half .. +31 of S
        const int quarter = warp & 3;                      // TMEM lanes 32 quarter .. +31
        const int r = quarter * 32 + lane;                 // query row of this thread
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const int pair_bar = 1 + quarter;
        const float sl = p.scale_log2;
        // waits do not change the control flow (the pair barriers must stay
        // matched); after an abort they return at once and the results are
        // discarded
        auto wait_all = [&](int which, uint32_t parity, int tag) {
            __syncwarp();
            mbar_wait(bar(which), parity, abort_flag, p.err, kErrWait, p.diag, tag);
            __syncwarp();
        };
        // the common case, a phase that has completed: one probe per lane and
        // a vote (338 against 342 µs a layer at long with the loop every time)
        auto wait_fast = [&](int which, uint32_t parity, int tag) {
            if (!__all_sync(0xffffffffu, mbar_try_wait(bar(which), parity))) wait_all(which, parity, tag);
        };
        // Q tile of query tile t into TMEM: this thread's half of row r (D / 2
        // bf16 = D / 4 columns); rows past the character's tail are zero
        auto stage_q = [&](int t) {
            grid_dependency_wait();                        // q_rot comes from the previous grid
            const Tile T = decode_tile(p, t);
            const AttnChar& ch = p.ch[T.b];
            const int tok = T.tok0 + r / g;
            constexpr int W = D / 4;                       // 32-bit words of this half
            uint4 v[W / 4];
            const uint4* src = reinterpret_cast<const uint4*>(
                p.q_rot + ((int64_t)(ch.tail_off + tok) * p.Hq + T.kvh * g + (r % g)) * D + half * (D / 2));
#pragma unroll
            for (int e = 0; e < W / 4; ++e) v[e] = tok < ch.M ? src[e] : make_uint4(0, 0, 0, 0);
            const uint32_t* w = reinterpret_cast<const uint32_t*>(v);
            if constexpr (W >= 32) {
#pragma unroll
                for (int c0 = 0; c0 < W; c0 += 32) {
                    uint32_t x[32];
#pragma unroll
                    for (int e = 0; e < 32; ++e) x[e] = w[c0 + e];
                    tmem_st32(tmem + lane_off + C::TMEM_Q + half * W + c0, x);
                }
            } else {
                uint32_t x[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) x[e] = w[e];
                tmem_st16(tmem + lane_off + C::TMEM_Q + half * W, x);
            }
            tmem_st_wait();
            tc_fence_before();
            mbar_arrive(bar(Q_FULL));
        };
        if (more(t_begin, k_begin)) stage_q(t_begin);
        int j = 0, seg = 0;
        for (int t = t_begin, k = k_begin; more(t, k); ++t, k = 0, ++seg) {
            const Tile T = decode_tile(p, t);
            const AttnChar& ch = p.ch[T.b];
            const int k1 = (t == t_end) ? k_end : T.nk;
            const int n = k1 - k;
            const bool full = (k == 0 && k1 == T.nk);
            const bool has_next = more(t + 1, 0);
            const int tok = T.tok0 + r / g;
            const bool row_valid = tok < ch.M;
            const int lim = ch.L_prev + min(tok, ch.M - 1) + 1;    // keys [0, lim) are visible
            float mr = -INFINITY;                        // reference max, log2 units
            float l = 0.f;                               // this half's share of the row sum
            for (int i = 0; i < n; ++i, ++j) {
                const int sb = j & 1;
                wait_fast(S_FULL + sb, (j >> 1) & 1, 0x31 + 256 * j);
                tc_fence_after();
                uint32_t sa[32];
                tmem_ld32(tmem + lane_off + C::TMEM_S + sb * BN + 32 * half, sa);
                tmem_ld_wait();
                tc_fence_before();
                mbar_arrive(bar(S_EMPTY + sb));
                // the segment's last S has landed, so no MMA reads Q any more
                if (i + 1 == n && has_next) stage_q(t + 1);
                const int key0 = (k + i) * BN + 32 * half;
                float s[32];
#pragma unroll
                for (int c = 0; c < 32; ++c) s[c] = __uint_as_float(sa[c]);
                if (key0 + 32 > lim) {
#pragma unroll
                    for (int c = 0; c < 32; ++c)
                        if (key0 + c >= lim) s[c] = -INFINITY;
                }
                float m16[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) m16[c] = fmaxf(s[c], s[c + 16]);
#pragma unroll
                for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
                    for (int c = 0; c < w; ++c) m16[c] = fmaxf(m16[c], m16[c + w]);
                const float pm = m16[0];
                float* xs = xch + sb * 2 * BM;           // [half][row] of this tile
                xs[half * BM + r] = pm;
                named_bar_sync(pair_bar, 64);
                const float mx2 = fmaxf(pm, xs[(1 - half) * BM + r]) * sl;
                const bool bump = mx2 > mr + 8.0f;       // also true while mr = -inf and a key is visible
                const float mr_new = bump ? mx2 : mr;
                float pv[32];
                float sum = 0.f;
                if (mr_new == -INFINITY) {
#pragma unroll
                    for (int c = 0; c < 32; ++c) pv[c] = 0.f;
                } else {
#pragma unroll
                    for (int c = 0; c < 32; ++c) pv[c] = ex2(fmaf(s[c], sl, -mr_new));
                    float a16[16];
#pragma unroll
                    for (int c = 0; c < 16; ++c) a16[c] = pv[c] + pv[c + 16];
#pragma unroll
                    for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
                        for (int c = 0; c < w; ++c) a16[c] += a16[c + w];
                    sum = a16[0];
                }
                const float factor = bump ? ((mr == -INFINITY) ? 0.f : ex2(mr - mr_new)) : 1.f;
                // P buffer sb is free once PV_{j-2} has completed
                if (j >= 2) wait_fast(PV_DONE + sb, ((j >> 1) - 1) & 1, 0x32 + 256 * j);
                if (i > 0 && __any_sync(0xffffffffu, bump)) {
                    // rescale this half of the O row once PV_{j-1} has landed
                    wait_all(PV_DONE + (sb ^ 1), ((j - 1) >> 1) & 1, 0x33 + 256 * j);
                    tc_fence_after();
#pragma unroll 1
                    for (int c0 = half * C::HALF; c0 < (half + 1) * C::HALF; c0 += 32) {
                        uint32_t o[32];
                        tmem_ld32(tmem + lane_off + C::TMEM_O + c0, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * factor);
                        tmem_st32(tmem + lane_off + C::TMEM_O + c0, o);
                    }
                    tmem_st_wait();
                }
                l = l * factor + sum;
                mr = mr_new;
                // 32 bf16 of row r = 16-byte chunks 4 half .. 4 half + 3, chunk index XOR (r & 7)
                const uint32_t prow = sP + sb * C::P_BYTES + r * 128;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        __nv_bfloat162 h2 = __floats2bfloat162_rn(pv[8 * q + 2 * e], pv[8 * q + 2 * e + 1]);
                        w[e] = *reinterpret_cast<uint32_t*>(&h2);
                    }
                    st_shared_v4(prow + (((4 * half + q) ^ (r & 7)) << 4), w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(bar(P_FULL + sb));
            }
            // ---------------------------------------------------------------- epilogue of the segment
            wait_all(O_FINAL, seg & 1, 0x34 + 256 * seg);
            tc_fence_after();
            float* xl = xch + (j & 1) * 2 * BM;          // the exchange buffer the last tile did not use
            xl[half * BM + r] = l;
            named_bar_sync(pair_bar, 64);
            const float lt = l + xl[(1 - half) * BM + r];
            named_bar_sync(pair_bar, 64);                // the buffer is free for the next segment
            const bool store = *abort_flag == 0;
            const int hq = T.kvh * g + (r % g);
            if (full) {
                // tcgen05.ld is warp-collective: every lane loads, real rows store
                const float inv = row_valid ? 1.f / lt : 0.f;
                __nv_bfloat16* o = p.out + ((int64_t)(ch.tail_off + (row_valid ? tok : 0)) * p.Hq + hq) * D;
#pragma unroll 1
                for (int c0 = half * C::HALF; c0 < (half + 1) * C::HALF; c0 += 32) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + C::TMEM_O + c0, v);
                    tmem_ld_wait();
                    if (row_valid && store) {
                        uint32_t w[16];
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            __nv_bfloat162 h2 = __floats2bfloat162_rn(__uint_as_float(v[2 * e]) * inv,
                                                                      __uint_as_float(v[2 * e + 1]) * inv);
                            w[e] = *reinterpret_cast<uint32_t*>(&h2);
                        }
                        uint4* dst = reinterpret_cast<uint4*>(o + c0);
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            dst[e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
                    }
                }
            } else {
                const int64_t prow = (int64_t)(2 * cta + (seg == 0 ? 0 : 1)) * BM + r;
                if (half == 0 && store) {
                    p.part_ml[prow * 2 + 0] = mr;
                    p.part_ml[prow * 2 + 1] = lt;
                }
                // partial layout [slot][D / 32][8][row][4]: each 16-byte store
                // of a warp lands in 512 contiguous bytes
                const int64_t slot = 2 * cta + (seg == 0 ? 0 : 1);
#pragma unroll 1
                for (int c0 = half * C::HALF; c0 < (half + 1) * C::HALF; c0 += 32) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + C::TMEM_O + c0, v);
                    tmem_ld_wait();
                    if (store) {
                        uint4* dst = reinterpret_cast<uint4*>(p.part_o + (slot * (D / 32) + c0 / 32) * 8 * BM * 4) + r;
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            dst[e * BM] = make_uint4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(bar(O_EMPTY));
        }
    }
    tc_fence_before();
    __syncthreads();
    if ((warp == 0 || warp == kVWarp) && lane == 0 && *abort_flag) {
        // copies still in flight land before the block releases its shared memory
        volatile int never = 0;
        const int full = warp == 0 ? K_FULL : V_FULL;
        for (int s = 0; s < STAGES; ++s)
            if (last_load[s] >= 0)
                mbar_wait(bar(full + s), (last_load[s] / STAGES) & 1, &never, p.err, kErrWait, nullptr, 0, 100000000ull);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

template <int D>
void launch_tc(const AttnParams& p, cudaStream_t s) {
    using C = Cfg<D>;
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(tail_attention_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        configured |= 1ull << (dev & 63);
    }
    launch_pdl(tail_attention_tc_kernel<D>, dim3(p.n_ctas), dim3(kThreads), C::SMEM, s, p);
}

}  // namespace

void launch_tail_attention(const AttnParams& p, cudaStream_t s) {
    if (p.n_ctas <= 0) return;
    switch (p.D) {
        case 64: launch_tc<64>(p, s); break;
        case 128: launch_tc<128>(p, s); break;
        case 256: launch_tc<256>(p, s); break;
        default: break;   // rejected on the host
    }
}

// One block per SM: 384 threads of about 150 registers leave no room for a
// second (and head_dim 256 needs all of TMEM and shared memory).
int attention_ctas_per_sm(int) { return 1; }

}  // namespace kvm
