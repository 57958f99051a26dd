// Gated delta rule from the carried state on the sm_100-family tensor cores
// (Eq. 3 for a recurrent layer; Gated DeltaNet, the layer family of §4.1):
//     S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T,  o_t = S_t q_t.
//
// Chunks of C = 64 tail tokens.  With g_t = sum_{u<=t} log alpha_u (within the
// chunk), G_t = exp(g_t) and w_j = beta_j exp(g_C - g_j):
//   KK, QK   = [K;Q] K^T
//   L        = strict_lower(exp(g_t - g_j) beta_j KK),  A = lower(exp(g_t - g_j) beta_j QK)
//   X        = [I; A] (I + L)^-1 = [T; A T]
//   W  = T G K,  U = T V,  A W,  A U                    (= X G K and X V)
//   Q' = G Q - A W
//   E  = U - W S0^T,   O = A U + Q' S0^T               (= G Q S0^T + A E)
//   S^T = G_C S0^T + K^T diag(w) E
// Everything above the line "E = ..." is independent of the state, so it runs
// in a prep kernel with one block of 512 threads per (chunk, head) (two when
// both fit on the SMs: one writes [W; Q'] and K, the other U | A U), all
// chunks in parallel;
// it leaves per (chunk, head) a record with [W; Q'] and K as ready-made MMA
// operand images, U and A U in fp32, w and G_C.  The scan kernel then walks
// the chunks of each (character, head, d_v slice) in order with the state in
// TMEM: each of the next record's images is fetched by one bulk copy as soon
// as the current one has been consumed; the MMA [W; Q'] S0^T, E and O, and
// the state update follow, with four block barriers per chunk.
//
// Tensor-core operands are bf16.  K, Q, V are exact in bf16 and used in place
// (K and V as MN-major operands in their natural row layout).  Every computed
// fp32 operand x (X, W, Q', S, w E) is split into x_hi = bf16(x) and
// x_lo = bf16(x - x_hi); a product with a split operand is hi*hi + hi*lo +
// lo*hi (or hi + lo against an exact operand) with fp32 accumulation, about
// 2^-15 relative accuracy.  The master state stays fp32 in TMEM.
#include <algorithm>

#include "kvm_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvm {
namespace {

using namespace ptx;

constexpr int C = 64;            // chunk length
constexpr int kThreads = 256;
constexpr int DVMAX = 128;       // d_v rows per scan block
constexpr int DVP = 256;         // largest d_v the prep kernel stages
constexpr int LSTRIDE = 68;      // fp32 row stride of the L scratch (conflict-free row vectors)
constexpr int DSTRIDE = 20;      // fp32 row stride of the diagonal-block inverses

// Workspace record of one (chunk, head):
//   [W;Q'] hi | [W;Q'] lo   (128 x DK bf16 each, K-major 128-byte-swizzled image)
//   K                       (64 x DK bf16, 128-byte-swizzled image, rows = tokens)
//   U | A U                 (fp32, rows 0..63 U, 64..127 A U, in slices of 32
//                            columns [dv/32][128][32]: a scan block's d_v rows are
//                            one contiguous piece; within a slice the 16-byte
//                            chunk c of row r sits at chunk (c + r) mod 8, so
//                            row-parallel reads of a copy in shared memory do not
//                            collide on banks)
//   w[64], G_C              (fp32)
template <int DK>
struct Rec {
    static constexpr int64_t WQH = 128 * DK * 2;
    static constexpr int64_t KIMG = 64 * DK * 2;
    static constexpr int64_t IMG = 2 * WQH + KIMG;
    static __host__ __device__ int64_t uau_off() { return IMG; }
    static __host__ __device__ int64_t misc_off(int dv) { return IMG + (int64_t)128 * dv * 4; }
    static __host__ __device__ int64_t bytes(int dv) { return IMG + (int64_t)128 * dv * 4 + 512; }
};

// Float offset of (row, col) in a U | A U copy of 32-column slices.
__device__ __forceinline__ int uau_idx(int row, int col) {
    return ((col >> 5) * 128 + row) * 32 + 4 * ((((col & 31) >> 2) + row) & 7) + (col & 3);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

// Split 8 fp32 values into bf16 hi and lo halves (8 bf16 each).
__device__ __forceinline__ void split8(const float* x, uint4& hi, uint4& lo) {
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 hh = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
        const float2 hf = __bfloat1622float2(hh);
        hw[e] = *reinterpret_cast<const uint32_t*>(&hh);
        lw[e] = pack_bf16x2(x[2 * e] - hf.x, x[2 * e + 1] - hf.y);
    }
    hi = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    lo = make_uint4(lw[0], lw[1], lw[2], lw[3]);
}

__device__ __forceinline__ int find_char_by_chunk(const GdnParams& p, int chunk) {
    int lo = 0, hi = p.n_chars - 1;              // last b with chunk_off <= chunk
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].chunk_off <= chunk) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// ============================================================================
// prep: one block of 512 threads per (chunk, head) (or two, see prep_parts)
// ============================================================================
constexpr int kPrepThreads = 512;

template <int DK>
struct PrepCfg {
    static constexpr int KQ = 128 * DK * 2;                  // [K;Q] bf16, K-major, 128 rows
    static constexpr int V = C * DVP * 2;                    // V bf16, rows j (MN-major operand)
    static constexpr int TILE128 = 128 * 64 * 2;             // 128 x 64 bf16 K-major tile
    static constexpr int LA = 64 * LSTRIDE * 4;              // fp32 [64][LSTRIDE]
    static constexpr int OFF_KQ = 0;
    static constexpr int OFF_V = OFF_KQ + KQ;
    static constexpr int OFF_L = OFF_V + V;                  // L (strictly lower), fp32
    static constexpr int OFF_XG = OFF_L + 2 * LA;            // [I; A] hi, lo, then X G hi, lo
    static constexpr int OFF_X = OFF_XG + 2 * TILE128;       // T hi, lo (MN-major), then X hi, lo
    static constexpr int OFF_D = OFF_X + 2 * TILE128;        // fp32 [64][DSTRIDE]: inverses of the diagonal blocks
    static constexpr int OFF_BAR = OFF_D + 64 * DSTRIDE * 4;
    static constexpr int SMEM = OFF_BAR + 64 + 1024;
    // record staging: [W;Q'] hi | lo over XG, X; U | A U over V, L
    static constexpr int OFF_STAGE_WQ = OFF_XG;
    static constexpr int OFF_STAGE_U = OFF_V;
    static_assert(OFF_XG % 1024 == 0, "operand tiles on 1024-byte boundaries");
    static_assert(2 * 128 * DK * 2 <= 4 * TILE128, "[W;Q'] staging");
    static_assert(128 * 128 * 4 <= V + 2 * LA, "U | A U staging for d_v <= 128");  // over V and L
    static constexpr uint32_t T_D = 0;                       // KK / QK (64 cols)
    static constexpr uint32_t T_WU = 128;                    // [W | U] (DK + dv cols)
};

// ============================================================================
// v2 (d_k = 128): the chain carries only the state.  Per chunk, with the
// state S0 entering it,
//     S^T = P_c S0^T + B_c,   P_c = G_C I - K^T diag(w) W,   B_c = K^T diag(w) U
// (the state update of the WY form with E = U - W S0^T substituted), and the
// outputs O = A U + Q' S0^T depend on S0 only through the chunk's snapshot.
// The prep forms P_c (hi | lo, the chain's K-major A operand) and B_c beside
// Q' and A U; the chain kernel runs one MMA batch and a refresh per chunk and
// writes each chunk's entering state as a snapshot; the output kernel then
// forms every chunk's outputs at once.
// ============================================================================
template <int DK>
struct Rec2 {
    static constexpr int64_t WQH = 128 * DK * 2;             // one half of the P_c image (128 rows)
    static constexpr int64_t QH = 64 * DK * 2;               // one half of the Q' image (64 rows)
    static __host__ __device__ int64_t pi_off() { return 0; }
    static __host__ __device__ int64_t qi_off() { return 2 * WQH; }
    static __host__ __device__ int64_t bc_off() { return 2 * WQH + 2 * QH; }
    static __host__ __device__ int64_t au_off(int dv) { return bc_off() + (int64_t)128 * dv * 4; }
    static __host__ __device__ int64_t bytes(int dv) { return au_off(dv) + (int64_t)64 * dv * 4; }
};

// Float offset of (row, col) in an A U copy of 32-column slices [dv/32][64][32].
__device__ __forceinline__ int au_idx(int row, int col) { return ((col >> 5) * 64 + row) * 32 + (col & 31); }

template <int DK>
struct Prep2Cfg {
    using G = PrepCfg<DK>;
    static constexpr uint32_t WW_HALF = 64 * DK * 2;         // w W operand half [64 tokens][DK]
    static constexpr uint32_t WU_HALF = 64 * 128 * 2;        // w U operand half [64 tokens][dv <= 128]
    static constexpr uint32_t OFF_WW = G::OFF_XG;            // over the X G tiles (consumed)
    static constexpr uint32_t OFF_WU = G::OFF_X;             // over the X tiles (consumed)
    static constexpr uint32_t OFF_QI = G::OFF_V;             // Q' staging over V (consumed)
    static constexpr uint32_t OFF_AU = G::OFF_L;             // A U staging over L (consumed)
    static constexpr uint32_t OFF_PI = G::OFF_XG;            // P_c staging once w W, w U are consumed
    static constexpr uint32_t OFF_BC = G::OFF_KQ;            // B_c staging over [K;Q], V, L
    static constexpr uint32_t T_P = 0;                       // P' (DK columns)
    static constexpr uint32_t T_B = 384;                     // B_c (dv columns)
    static_assert(2 * WW_HALF <= 2 * G::TILE128 && 2 * WU_HALF <= 2 * G::TILE128, "operand staging");
    static_assert(2 * 64 * DK * 2 <= G::V, "Q' staging");
    static_assert(64 * 128 * 4 <= 2 * G::LA, "A U staging");
    static_assert(2 * 128 * DK * 2 <= 4 * G::TILE128, "P_c staging");
    static_assert(128 * 128 * 4 <= G::OFF_XG - G::OFF_KQ, "B_c staging");
};


// Fused launches (gdn_fused_kernel): a finished record is published by
// setting its flag to the launch's epoch; the scan waits for it.  Standalone
// launches pass flags = null (the records complete with the prep grid).
struct FuseCtl {
    uint32_t* flags;      // [record][kFlagWords], record = chunk * H + head
    uint32_t epoch;
};
constexpr int kFlagWords = 32;   // one flag per 128-byte line

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release_u32(uint32_t* p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Orders this thread's async-proxy (bulk copy) accesses of global memory
// with its generic-proxy ones.
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Record `rec` (chunk * H + head) of a fused launch: wait (one thread,
// bounded in wall time) until the prep has published it, then order the
// bulk copies that follow after that observation.
__device__ __forceinline__ bool wait_record(const FuseCtl& fc, int64_t rec, volatile int* abort_flag, int* err,
                                            int* diag, int tag) {
    if (!fc.flags) return true;
    const uint32_t* f = fc.flags + rec * kFlagWords;
    uint64_t t0 = 0;
    for (uint32_t it = 0;; ++it) {
        if (ld_acquire_u32(f) == fc.epoch) {
            fence_proxy_async_global();
            return true;
        }
        if ((it & 15) == 15) {
            if (*abort_flag) return false;
            const uint64_t now = globaltimer_ns();
            if (t0 == 0) t0 = now;
            else if (now - t0 > 250000000ull) {
                *abort_flag = 1;
                atomicOr(err, kErrWait);
                if (diag && atomicCAS(diag, 0, (int)blockIdx.x + 1) == 0) {
                    diag[1] = tag;
                    diag[2] = 0;
                }
                return false;
            }
        }
        __nanosleep(32);
    }
}

// Work unit u of a fused launch's prep workers: units are ordered by the
// chunk's index within its character, then character, then head, so that
// every character's scan finds its next chunk ready early.  Returns
// chunk * H + head, or -1 past the last unit.
__device__ __forceinline__ int fused_unit(const GdnParams& p, int u) {
    for (int i = 0;; ++i) {
        bool any = false;
        for (int b = 0; b < p.n_chars; ++b) {
            if ((p.ch[b].M + C - 1) / C > i) {
                if (u < p.H) return (p.ch[b].chunk_off + i) * p.H + u;
                u -= p.H;
                any = true;
            }
        }
        if (!any) return -1;
    }
}

// The prep's work units u = u0, u0 + ustride, ... (standalone: one unit per
// block, u = blockIdx.x over (chunk, head, part); fused: the units of
// fused_unit, one part each).
template <int DK>
__device__ __forceinline__ void gdn_prep_run(const GdnParams& p, const FuseCtl& fc, int u0, int ustride) {
    using G = PrepCfg<DK>;
    using R = Rec<DK>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oKQ = G::OFF_KQ, oV = G::OFF_V, oXG = G::OFF_XG, oX = G::OFF_X;
    constexpr uint32_t T128 = G::TILE128;
    float* Lm = reinterpret_cast<float*>(smem + G::OFF_L);
    uint64_t* bar = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 8);
    const uint32_t mbar = smem_u32(bar);
    __shared__ float gs[C], bs[C], Gs[C], g2[C];
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, cq = warp >> 2;         // TMEM lane quarter, column quarter
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int H = p.H, dv = p.dv;
    const int parts = fc.flags ? 1 : p.prep_parts;
    const int n_units = p.total_chunks * H * parts;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    grid_dependency_wait();                          // the chunk inputs may come from the previous grid
    grid_dependents_launch();
    uint32_t phase = 0;
    for (int u = u0; u < n_units; u += ustride) {
    // with two parts per (chunk, head) both solve for X; part 0 writes the
    // [W; Q'] and K images, part 1 U | A U and w, G_C
    const int part = u % parts;
    const int ch_h = fc.flags ? fused_unit(p, u) : u / parts;
    if (ch_h < 0) break;                             // uniform per block (not reached for valid grids)
    const bool do_w = parts == 1 || part == 0;
    const bool do_u = parts == 1 || part == 1;
    const int chunk = ch_h / H, h = ch_h % H;
    const int b = find_char_by_chunk(p, chunk);
    const GdnChar ch = p.ch[b];
    const int c0 = (chunk - ch.chunk_off) * C;
    if (c0 >= ch.M) continue;                        // uniform per block (not reached for valid grids)
    const int n = min(C, ch.M - c0);
    const int64_t tok0 = ch.tail_off + c0;
    uint8_t* rec = p.work + ((int64_t)chunk * H + h) * p.rec_bytes;
    // ---- loads (every global load issued before the shared stores)
    {
        constexpr int NKQ = 128 * (DK / 8) / kPrepThreads;
        constexpr int NV = C * (DVP / 8) / kPrepThreads;
        uint4 kq[NKQ], vv[NV];
#pragma unroll
        for (int u = 0; u < NKQ; ++u) {
            const int i = tid + u * kPrepThreads;
            const int rr = i / (DK / 8), c8 = (i % (DK / 8)) * 8, t = rr & 63;
            kq[u] = t < n ? __ldg(reinterpret_cast<const uint4*>((rr < 64 ? p.k : p.q) + ((tok0 + t) * H + h) * DK + c8))
                          : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int i = tid + u * kPrepThreads;
            const int t = i / (dv / 8), r8 = (i % (dv / 8)) * 8;
            vv[u] = (do_u && i < C * (dv / 8) && t < n) ? __ldg(reinterpret_cast<const uint4*>(p.v + ((tok0 + t) * H + h) * dv + r8))
                                                : make_uint4(0, 0, 0, 0);
        }
        // the gates of the chunk (warp 0)
        float a0 = 1.f, a1 = 1.f, b0 = 0.f, b1 = 0.f;
        if (tid < 32) {
            if (tid < n) { a0 = __ldg(p.alpha + (tok0 + tid) * H + h); b0 = __ldg(p.beta + (tok0 + tid) * H + h); }
            if (tid + 32 < n) { a1 = __ldg(p.alpha + (tok0 + tid + 32) * H + h); b1 = __ldg(p.beta + (tok0 + tid + 32) * H + h); }
        }
#pragma unroll
        for (int u = 0; u < NKQ; ++u) {
            const int i = tid + u * kPrepThreads;
            const int rr = i / (DK / 8), c8 = (i % (DK / 8)) * 8;
            V4(oKQ + sw128_off16(rr, c8, 128)) = kq[u];
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int i = tid + u * kPrepThreads;
            if (do_u && i < C * (dv / 8)) V4(oV + sw128_off16(i / (dv / 8), (i % (dv / 8)) * 8, C)) = vv[u];
        }
        if (tid < 32) {
            float x0 = tid < n ? logf(a0) : 0.f;
            float x1 = tid + 32 < n ? logf(a1) : 0.f;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y0 = __shfl_up_sync(0xffffffffu, x0, o);
                const float y1 = __shfl_up_sync(0xffffffffu, x1, o);
                if (tid >= o) { x0 += y0; x1 += y1; }
            }
            x1 += __shfl_sync(0xffffffffu, x0, 31);
            gs[tid] = x0;
            gs[tid + 32] = x1;
            bs[tid] = b0;
            bs[tid + 32] = b1;
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    if (tid < C) {
        Gs[tid] = expf(gs[tid]);
        g2[tid] = gs[tid] * 1.4426950408889634f;          // log2 domain for the decays
        if (do_u) {
            float* misc = reinterpret_cast<float*>(rec + R::misc_off(dv));
            misc[tid] = tid < n ? bs[tid] * expf(gs[n - 1] - gs[tid]) : 0.f;     // w_j
            if (tid == 0) misc[C] = expf(gs[n - 1]);                            // G_C
        }
    }
    bool ok = true;
    // the issuing thread waits for its MMAs and the block follows it at the
    // barrier (waiting lanes of the issuer's warp would slow its issue)
    auto mma_wait = [&]() -> bool {
        bool r = true;
        if (tid == 0) r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait, p.diag, 0x40);
        phase ^= 1;
        r = __syncthreads_and(r);
        tc_fence_after();
        return r;
    };
    const uint32_t kq_region = 128 * 128;
    // ---------------------------------------------------------------- KK, QK
    if (tid == 0) {
#pragma unroll
        for (int ks = 0; ks < DK / 16; ++ks) {
            const uint32_t off = (ks >> 2) * kq_region + (ks & 3) * 32;
            mma_bf16(tmem + G::T_D, smem_desc_sw128(sb + oKQ + off, 16, 1024), smem_desc_sw128(sb + oKQ + off, 16, 1024),
                     idesc_bf16_f32(128, C, false), ks > 0);
        }
        mma_commit(mbar);
        if (do_w) {
            // the K image (rows 0..63 of each 64-column region of [K;Q]) is
            // final already; it leaves now, beside the rest of the kernel
            for (int r = 0; r < DK / 64; ++r)
                bulk_store(rec + 2 * R::WQH + r * (64 * 128), sb + oKQ + r * (128 * 128), 64 * 128);
            bulk_commit();
        }
    }
    ok = mma_wait();                                // also publishes Gs
    // ---------------------------------------------------------------- L (rows < 64), A (rows >= 64)
    // L goes to shared memory in fp32 for the solve of T = (I + L)^-1; the
    // rows of [I; A] go straight into the A operand of X = [I; A] T (bf16 hi |
    // lo, K-major, over the XG tiles).  Thread (row, cq) forms columns
    // 16 cq .. 16 cq + 15 of TMEM row `row`.
    if (ok) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_off + G::T_D + cq * 16, v);
        tmem_ld_wait();
        const int t = row & 63;
        const float gt2 = g2[t];
        float y[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            const int j = cq * 16 + c;
            const bool keep = (row < 64) ? (j < t) : (j <= t);
            y[c] = (keep && t < n) ? ex2(gt2 - g2[j]) * bs[j] * __uint_as_float(v[c]) : 0.f;
        }
        if (row < 64) {
            float* dst = Lm + t * LSTRIDE + cq * 16;
#pragma unroll
            for (int j4 = 0; j4 < 16; j4 += 4) *reinterpret_cast<float4*>(dst + j4) = make_float4(y[j4], y[j4 + 1], y[j4 + 2], y[j4 + 3]);
#pragma unroll
            for (int c = 0; c < 16; ++c) y[c] = (cq * 16 + c == row) ? 1.f : 0.f;     // row of I
        }
#pragma unroll
        for (int j8 = 0; j8 < 16; j8 += 8) {
            uint4 hi, lo;
            split8(y + j8, hi, lo);
            const uint32_t off = sw128_off16(row, cq * 16 + j8, 128);
            V4(oXG + off) = hi;
            V4(oXG + T128 + off) = lo;
        }
    }
    __syncthreads();
    // ---------------------------------------------------------------- T = (I + L)^-1
    // With I + L cut into 16 x 16 blocks (lower triangular by blocks, D_j the
    // inverse of diagonal block j), row p of T solves x (I + L) = e_p column
    // block by column block from the right: x_j = (b_j - sum_{i > j} x_i L_ij) D_j,
    // zero right of column p.  The D_j come first (thread t < 64 solves
    // column t mod 16 of block t / 16).
    float* Dm = reinterpret_cast<float*>(smem + G::OFF_D);
    if (ok && tid < 64) {
        const int kb = tid >> 4, c = tid & 15;
        float d[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float* li = Lm + (16 * kb + i) * LSTRIDE + 16 * kb;
            float v = (i == c) ? 1.f : 0.f;
#pragma unroll
            for (int m = 0; m < i; ++m) v = fmaf(-li[m], d[m], v);
            d[i] = v;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) Dm[(16 * kb + i) * DSTRIDE + c] = d[i];
    }
    __syncthreads();
    // Eight threads per row pr (tid = 8 pr + q); thread q owns columns
    // 16 k + 2 q, 16 k + 2 q + 1 of every block k; warps (four rows of one
    // block) skip the blocks right of it.  T leaves as the B operand
    // (MN-major, rows = the contraction index) of X = [I; A] T, bf16 hi | lo
    // over the X tiles.
    if (ok) {
        const int pr = tid >> 3, q = tid & 7;
        float xs[8];                                  // xs[2k + e] = x[16k + 2q + e]
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int e = 0; e < 2; ++e) xs[2 * k + e] = (16 * k + 2 * q + e == pr) ? 1.f : 0.f;
        const int top = pr >> 4;                      // uniform per warp (four rows of one block)
#pragma unroll
        for (int jb = 3; jb >= 0; --jb) {
            if (jb > top) continue;
            // yv[o][e] = current x[16 jb + 2 (q ^ o) + e]
            float yv[8][2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float a = xs[2 * jb + e];
                yv[0][e] = a;
#pragma unroll
                for (int o = 1; o < 8; ++o) yv[o][e] = __shfl_xor_sync(0xffffffffu, a, o);
            }
            float xb[2] = {0.f, 0.f};
#pragma unroll
            for (int o = 0; o < 8; ++o)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float2 d2 = *reinterpret_cast<const float2*>(Dm + (16 * jb + 2 * (q ^ o) + e) * DSTRIDE + 2 * q);
                    xb[0] = fmaf(yv[o][e], d2.x, xb[0]);
                    xb[1] = fmaf(yv[o][e], d2.y, xb[1]);
                }
            float xv[8][2];
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                xs[2 * jb + c] = xb[c];
                xv[0][c] = xb[c];
#pragma unroll
                for (int o = 1; o < 8; ++o) xv[o][c] = __shfl_xor_sync(0xffffffffu, xb[c], o);
            }
#pragma unroll
            for (int kb = 0; kb < jb; ++kb)
#pragma unroll
                for (int o = 0; o < 8; ++o)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const float2 l2 = *reinterpret_cast<const float2*>(
                            Lm + (16 * jb + 2 * (q ^ o) + e) * LSTRIDE + 16 * kb + 2 * q);
                        xs[2 * kb + 0] = fmaf(-xv[o][e], l2.x, xs[2 * kb + 0]);
                        xs[2 * kb + 1] = fmaf(-xv[o][e], l2.y, xs[2 * kb + 1]);
                    }
        }
        // T row pr, columns 16 k + 2 q and + 1: 4 bytes of each of hi and lo
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const __nv_bfloat16 h0 = __float2bfloat16_rn(xs[2 * k]), h1 = __float2bfloat16_rn(xs[2 * k + 1]);
            const float f0 = __bfloat162float(h0), f1 = __bfloat162float(h1);
            const uint32_t off = sw128_off16(pr, 16 * k + 2 * q, 64);
            *reinterpret_cast<uint32_t*>(smem + oX + off) = pack_bf16x2(f0, f1);
            *reinterpret_cast<uint32_t*>(smem + oX + 64 * 128 + off) = pack_bf16x2(xs[2 * k] - f0, xs[2 * k + 1] - f1);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---------------------------------------------------------------- X = [I; A] T on the tensor cores
    if (ok && tid == 0) {
        tc_fence_after();
        const uint32_t id_x = idesc_bf16_f32(128, C, true);          // B = T, MN-major
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks) {
            const uint64_t a_hi = smem_desc_sw128(sb + oXG + ks * 32, 16, 1024);
            const uint64_t a_lo = smem_desc_sw128(sb + oXG + T128 + ks * 32, 16, 1024);
            const uint64_t b_hi = smem_desc_sw128(sb + oX + ks * 16 * 128, C * 128, 1024);
            const uint64_t b_lo = smem_desc_sw128(sb + oX + 64 * 128 + ks * 16 * 128, C * 128, 1024);
            mma_bf16(tmem + G::T_D, a_hi, b_hi, id_x, ks > 0);
            mma_bf16(tmem + G::T_D, a_hi, b_lo, id_x, 1u);
            mma_bf16(tmem + G::T_D, a_lo, b_hi, id_x, 1u);
        }
        mma_commit(mbar);
    }
    if (ok) ok = mma_wait();
    // operands: X G (for W) and X (for U), K-major rows, from TMEM
    if (ok) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_off + G::T_D + cq * 16, v);
        tmem_ld_wait();
#pragma unroll
        for (int j8 = 0; j8 < 16; j8 += 8) {
            float xr[8], xg[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                xr[e] = __uint_as_float(v[j8 + e]);
                xg[e] = xr[e] * Gs[cq * 16 + j8 + e];
            }
            uint4 hi, lo;
            const uint32_t off = sw128_off16(row, cq * 16 + j8, 128);
            if (do_w) {
                split8(xg, hi, lo);
                V4(oXG + off) = hi;
                V4(oXG + T128 + off) = lo;
            }
            if (do_u) {
                split8(xr, hi, lo);
                V4(oX + off) = hi;
                V4(oX + T128 + off) = lo;
            }
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---------------------------------------------------------------- [W | U] = X [G K | V]
    if (ok && tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks) {
            const uint64_t bk = smem_desc_sw128(sb + oKQ + ks * 2048, kq_region, 1024);
            const uint64_t bvv = smem_desc_sw128(sb + oV + ks * 2048, C * 128, 1024);
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {             // the hi and lo halves of the X operand
                const uint32_t ao = hl * T128 + ks * 32;
                if (do_w)
                    mma_bf16(tmem + G::T_WU, smem_desc_sw128(sb + oXG + ao, 16, 1024), bk,
                             idesc_bf16_f32(128, DK, true), (ks | hl) != 0);
                if (do_u)
                    mma_bf16(tmem + G::T_WU + DK, smem_desc_sw128(sb + oX + ao, 16, 1024), bvv,
                             idesc_bf16_f32(128, dv, true), (ks | hl) != 0);
            }
        }
        mma_commit(mbar);
    }
    if (ok) ok = mma_wait();
    // ---------------------------------------------------------------- record: [W; Q'] image, U | A U
    // Both are staged in shared memory in their record layout (the MMA
    // operands they overwrite are consumed), 64 columns at a time: thread
    // (row, cq) takes the 16-column piece cq of each, and each 64-column
    // piece leaves in bulk copies while the next one is staged ([W; Q'] keeps
    // 64-column regions, U | A U 32-column slices, so a piece is contiguous).
    {
        const int t = row & 63;
        const float gt = Gs[t];
        const uint32_t oWQ = G::OFF_STAGE_WQ;
        float* us = reinterpret_cast<float*>(smem + G::OFF_STAGE_U);
        const int n_w = do_w ? DK / 64 : 0;
        const int n_u = do_u ? (dv + 63) / 64 : 0;
        for (int k = 0; k < n_w + n_u; ++k) {            // uniform per block
            const bool w_piece = k < n_w;
            if (ok && w_piece) {
                const int cb = 64 * k + 16 * cq;
                uint32_t v[16];
                tmem_ld16(tmem + lane_off + G::T_WU + cb, v);
                tmem_ld_wait();
                float y[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) y[j] = __uint_as_float(v[j]);
                if (row >= 64) {
                    // Q' = G Q - A W ; row `row` of [K;Q] holds q_t
#pragma unroll
                    for (int j8 = 0; j8 < 16; j8 += 8) {
                        const uint4 q8 = V4(oKQ + sw128_off16(row, cb + j8, 128));
                        const uint32_t* qw = reinterpret_cast<const uint32_t*>(&q8);
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[e]));
                            y[j8 + 2 * e] = gt * f.x - y[j8 + 2 * e];
                            y[j8 + 2 * e + 1] = gt * f.y - y[j8 + 2 * e + 1];
                        }
                    }
                }
#pragma unroll
                for (int j8 = 0; j8 < 16; j8 += 8) {
                    uint4 hi, lo;
                    split8(y + j8, hi, lo);
                    const uint32_t off = sw128_off16(row, cb + j8, 128);
                    V4(oWQ + off) = hi;
                    V4(oWQ + (uint32_t)R::WQH + off) = lo;
                }
            } else if (ok) {
                const int rc = 64 * (k - n_w) + 16 * cq;
                if (rc < dv) {                           // uniform per warp
                    uint32_t v[16];
                    tmem_ld16(tmem + lane_off + G::T_WU + DK + rc, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int j4 = 0; j4 < 16; j4 += 4)
                        *reinterpret_cast<uint4*>(us + uau_idx(row, rc + j4)) = make_uint4(v[j4], v[j4 + 1], v[j4 + 2], v[j4 + 3]);
                }
            }
            fence_proxy_async_smem();
            __syncthreads();
            if (ok && tid == 0) {
                if (w_piece) {
                    bulk_store(rec + k * (128 * 128), sb + oWQ + k * (128 * 128), 128 * 128);
                    bulk_store(rec + R::WQH + k * (128 * 128), sb + oWQ + (uint32_t)R::WQH + k * (128 * 128), 128 * 128);
                } else {
                    const int u = k - n_w;                 // slices 2u, 2u + 1
                    const int slices = min(2, dv / 32 - 2 * u);
                    bulk_store(rec + R::uau_off() + (int64_t)u * 2 * (128 * 32 * 4),
                               sb + G::OFF_STAGE_U + u * 2 * (128 * 32 * 4), slices * (128 * 32 * 4));
                }
                bulk_commit();
            }
        }
        if (tid == 0) {
            // the sources must be read before the block's shared memory is
            // released or restaged; standalone, the writes complete with the
            // grid, before the scan (which waits on this grid) reads them
            bulk_wait_read();
        }
    }
    // fused: w and G_C (plain stores above) are ordered before the record's
    // flag; fencing here, long after the stores, costs little
    if (fc.flags && do_u && tid < C) __threadfence();
    tc_fence_before();
    __syncthreads();                                 // the staging area is free for the next unit
    tc_fence_after();
    if (fc.flags && tid == 0 && ok) {
        // fused: publish the record once its writes have completed (the
        // other threads are already loading the next unit)
        bulk_wait_all();
        fence_proxy_async_global();
        __threadfence();
        st_release_u32(fc.flags + (int64_t)ch_h * kFlagWords, fc.epoch);
    }
    }  // units
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(*tmem_slot, 512);
    }
}

template <int DK>
__global__ void __launch_bounds__(kPrepThreads, 1) gdn_prep_kernel(const __grid_constant__ GdnParams p) {
    gdn_prep_run<DK>(p, FuseCtl{nullptr, 0}, blockIdx.x, gridDim.x);
}

// v2 prep: the front (loads .. [W | U]) is the v1 prep's; the record differs.
template <int DK>
__device__ __forceinline__ void gdn_prep2_run(const GdnParams& p, const FuseCtl& fc, int u0, int ustride) {
    using G = PrepCfg<DK>;
    using G2 = Prep2Cfg<DK>;
    using R = Rec2<DK>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oKQ = G::OFF_KQ, oV = G::OFF_V, oXG = G::OFF_XG, oX = G::OFF_X;
    constexpr uint32_t T128 = G::TILE128;
    float* Lm = reinterpret_cast<float*>(smem + G::OFF_L);
    uint64_t* bar = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 8);
    const uint32_t mbar = smem_u32(bar);
    __shared__ float gs[C], bs[C], Gs[C], g2[C], ws[C];
    __shared__ float gC_sh;
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, cq = warp >> 2;         // TMEM lane quarter, column quarter
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int H = p.H, dv = p.dv;
    const int parts = 1;                             // v2: one block per (chunk, head)
    const int n_units = p.total_chunks * H * parts;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    if (!fc.flags) {                                 // the fused kernel waited already
        grid_dependency_wait();
        grid_dependents_launch();
    }
    uint32_t phase = 0;
    for (int u = u0; u < n_units; u += ustride) {
    // with two parts per (chunk, head) both solve for X; part 0 writes the
    // [W; Q'] and K images, part 1 U | A U and w, G_C
    const int part = u % parts;
    const int ch_h = fc.flags ? fused_unit(p, u) : u / parts;
    if (ch_h < 0) break;                             // uniform per block (not reached for valid grids)
    const bool do_w = parts == 1 || part == 0;
    const bool do_u = parts == 1 || part == 1;
    const int chunk = ch_h / H, h = ch_h % H;
    const int b = find_char_by_chunk(p, chunk);
    const GdnChar ch = p.ch[b];
    const int c0 = (chunk - ch.chunk_off) * C;
    if (c0 >= ch.M) continue;                        // uniform per block (not reached for valid grids)
    const int n = min(C, ch.M - c0);
    const int64_t tok0 = ch.tail_off + c0;
    uint8_t* rec = p.work + ((int64_t)chunk * H + h) * p.rec_bytes;
    // ---- loads (every global load issued before the shared stores)
    {
        constexpr int NKQ = 128 * (DK / 8) / kPrepThreads;
        constexpr int NV = C * (DVP / 8) / kPrepThreads;
        uint4 kq[NKQ], vv[NV];
#pragma unroll
        for (int u = 0; u < NKQ; ++u) {
            const int i = tid + u * kPrepThreads;
            const int rr = i / (DK / 8), c8 = (i % (DK / 8)) * 8, t = rr & 63;
            kq[u] = t < n ? __ldg(reinterpret_cast<const uint4*>((rr < 64 ? p.k : p.q) + ((tok0 + t) * H + h) * DK + c8))
                          : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int i = tid + u * kPrepThreads;
            const int t = i / (dv / 8), r8 = (i % (dv / 8)) * 8;
            vv[u] = (do_u && i < C * (dv / 8) && t < n) ? __ldg(reinterpret_cast<const uint4*>(p.v + ((tok0 + t) * H + h) * dv + r8))
                                                : make_uint4(0, 0, 0, 0);
        }
        // the gates of the chunk (warp 0)
        float a0 = 1.f, a1 = 1.f, b0 = 0.f, b1 = 0.f;
        if (tid < 32) {
            if (tid < n) { a0 = __ldg(p.alpha + (tok0 + tid) * H + h); b0 = __ldg(p.beta + (tok0 + tid) * H + h); }
            if (tid + 32 < n) { a1 = __ldg(p.alpha + (tok0 + tid + 32) * H + h); b1 = __ldg(p.beta + (tok0 + tid + 32) * H + h); }
        }
#pragma unroll
        for (int u = 0; u < NKQ; ++u) {
            const int i = tid + u * kPrepThreads;
            const int rr = i / (DK / 8), c8 = (i % (DK / 8)) * 8;
            V4(oKQ + sw128_off16(rr, c8, 128)) = kq[u];
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) {
            const int i = tid + u * kPrepThreads;
            if (do_u && i < C * (dv / 8)) V4(oV + sw128_off16(i / (dv / 8), (i % (dv / 8)) * 8, C)) = vv[u];
        }
        if (tid < 32) {
            float x0 = tid < n ? logf(a0) : 0.f;
            float x1 = tid + 32 < n ? logf(a1) : 0.f;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y0 = __shfl_up_sync(0xffffffffu, x0, o);
                const float y1 = __shfl_up_sync(0xffffffffu, x1, o);
                if (tid >= o) { x0 += y0; x1 += y1; }
            }
            x1 += __shfl_sync(0xffffffffu, x0, 31);
            gs[tid] = x0;
            gs[tid + 32] = x1;
            bs[tid] = b0;
            bs[tid + 32] = b1;
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    if (tid < C) {
        Gs[tid] = expf(gs[tid]);
        g2[tid] = gs[tid] * 1.4426950408889634f;          // log2 domain for the decays
        ws[tid] = tid < n ? bs[tid] * expf(gs[n - 1] - gs[tid]) : 0.f;         // w_j
        if (tid == 0) gC_sh = expf(gs[n - 1]);                                  // G_C
    }
    bool ok = true;
    // the issuing thread waits for its MMAs and the block follows it at the
    // barrier (waiting lanes of the issuer's warp would slow its issue)
    auto mma_wait = [&]() -> bool {
        bool r = true;
        if (tid == 0) r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait, p.diag, 0x40);
        phase ^= 1;
        r = __syncthreads_and(r);
        tc_fence_after();
        return r;
    };
    const uint32_t kq_region = 128 * 128;
    // ---------------------------------------------------------------- KK, QK
    if (tid == 0) {
#pragma unroll
        for (int ks = 0; ks < DK / 16; ++ks) {
            const uint32_t off = (ks >> 2) * kq_region + (ks & 3) * 32;
            mma_bf16(tmem + G::T_D, smem_desc_sw128(sb + oKQ + off, 16, 1024), smem_desc_sw128(sb + oKQ + off, 16, 1024),
                     idesc_bf16_f32(128, C, false), ks > 0);
        }
        mma_commit(mbar);
    }
    ok = mma_wait();                                // also publishes Gs
    // ---------------------------------------------------------------- L (rows < 64), A (rows >= 64)
    // L goes to shared memory in fp32 for the solve of T = (I + L)^-1; the
    // rows of [I; A] go straight into the A operand of X = [I; A] T (bf16 hi |
    // lo, K-major, over the XG tiles).  Thread (row, cq) forms columns
    // 16 cq .. 16 cq + 15 of TMEM row `row`.
    if (ok) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_off + G::T_D + cq * 16, v);
        tmem_ld_wait();
        const int t = row & 63;
        const float gt2 = g2[t];
        float y[16];
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            const int j = cq * 16 + c;
            const bool keep = (row < 64) ? (j < t) : (j <= t);
            y[c] = (keep && t < n) ? ex2(gt2 - g2[j]) * bs[j] * __uint_as_float(v[c]) : 0.f;
        }
        if (row < 64) {
            float* dst = Lm + t * LSTRIDE + cq * 16;
#pragma unroll
            for (int j4 = 0; j4 < 16; j4 += 4) *reinterpret_cast<float4*>(dst + j4) = make_float4(y[j4], y[j4 + 1], y[j4 + 2], y[j4 + 3]);
#pragma unroll
            for (int c = 0; c < 16; ++c) y[c] = (cq * 16 + c == row) ? 1.f : 0.f;     // row of I
        }
#pragma unroll
        for (int j8 = 0; j8 < 16; j8 += 8) {
            uint4 hi, lo;
            split8(y + j8, hi, lo);
            const uint32_t off = sw128_off16(row, cq * 16 + j8, 128);
            V4(oXG + off) = hi;
            V4(oXG + T128 + off) = lo;
        }
    }
    __syncthreads();
    // ---------------------------------------------------------------- T = (I + L)^-1
    // With I + L cut into 16 x 16 blocks (lower triangular by blocks, D_j the
    // inverse of diagonal block j), row p of T solves x (I + L) = e_p column
    // block by column block from the right: x_j = (b_j - sum_{i > j} x_i L_ij) D_j,
    // zero right of column p.  The D_j come first (thread t < 64 solves
    // column t mod 16 of block t / 16).
    float* Dm = reinterpret_cast<float*>(smem + G::OFF_D);
    if (ok && tid < 64) {
        const int kb = tid >> 4, c = tid & 15;
        float d[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float* li = Lm + (16 * kb + i) * LSTRIDE + 16 * kb;
            float v = (i == c) ? 1.f : 0.f;
#pragma unroll
            for (int m = 0; m < i; ++m) v = fmaf(-li[m], d[m], v);
            d[i] = v;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) Dm[(16 * kb + i) * DSTRIDE + c] = d[i];
    }
    __syncthreads();
    // Eight threads per row pr (tid = 8 pr + q); thread q owns columns
    // 16 k + 2 q, 16 k + 2 q + 1 of every block k; warps (four rows of one
    // block) skip the blocks right of it.  T leaves as the B operand
    // (MN-major, rows = the contraction index) of X = [I; A] T, bf16 hi | lo
    // over the X tiles.
    if (ok) {
        const int pr = tid >> 3, q = tid & 7;
        float xs[8];                                  // xs[2k + e] = x[16k + 2q + e]
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int e = 0; e < 2; ++e) xs[2 * k + e] = (16 * k + 2 * q + e == pr) ? 1.f : 0.f;
        const int top = pr >> 4;                      // uniform per warp (four rows of one block)
#pragma unroll
        for (int jb = 3; jb >= 0; --jb) {
            if (jb > top) continue;
            // yv[o][e] = current x[16 jb + 2 (q ^ o) + e]
            float yv[8][2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float a = xs[2 * jb + e];
                yv[0][e] = a;
#pragma unroll
                for (int o = 1; o < 8; ++o) yv[o][e] = __shfl_xor_sync(0xffffffffu, a, o);
            }
            float xb[2] = {0.f, 0.f};
#pragma unroll
            for (int o = 0; o < 8; ++o)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float2 d2 = *reinterpret_cast<const float2*>(Dm + (16 * jb + 2 * (q ^ o) + e) * DSTRIDE + 2 * q);
                    xb[0] = fmaf(yv[o][e], d2.x, xb[0]);
                    xb[1] = fmaf(yv[o][e], d2.y, xb[1]);
                }
            float xv[8][2];
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                xs[2 * jb + c] = xb[c];
                xv[0][c] = xb[c];
#pragma unroll
                for (int o = 1; o < 8; ++o) xv[o][c] = __shfl_xor_sync(0xffffffffu, xb[c], o);
            }
#pragma unroll
            for (int kb = 0; kb < jb; ++kb)
#pragma unroll
                for (int o = 0; o < 8; ++o)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const float2 l2 = *reinterpret_cast<const float2*>(
                            Lm + (16 * jb + 2 * (q ^ o) + e) * LSTRIDE + 16 * kb + 2 * q);
                        xs[2 * kb + 0] = fmaf(-xv[o][e], l2.x, xs[2 * kb + 0]);
                        xs[2 * kb + 1] = fmaf(-xv[o][e], l2.y, xs[2 * kb + 1]);
                    }
        }
        // T row pr, columns 16 k + 2 q and + 1: 4 bytes of each of hi and lo
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const __nv_bfloat16 h0 = __float2bfloat16_rn(xs[2 * k]), h1 = __float2bfloat16_rn(xs[2 * k + 1]);
            const float f0 = __bfloat162float(h0), f1 = __bfloat162float(h1);
            const uint32_t off = sw128_off16(pr, 16 * k + 2 * q, 64);
            *reinterpret_cast<uint32_t*>(smem + oX + off) = pack_bf16x2(f0, f1);
            *reinterpret_cast<uint32_t*>(smem + oX + 64 * 128 + off) = pack_bf16x2(xs[2 * k] - f0, xs[2 * k + 1] - f1);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---------------------------------------------------------------- X = [I; A] T on the tensor cores
    if (ok && tid == 0) {
        tc_fence_after();
        const uint32_t id_x = idesc_bf16_f32(128, C, true);          // B = T, MN-major
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks) {
            const uint64_t a_hi = smem_desc_sw128(sb + oXG + ks * 32, 16, 1024);
            const uint64_t a_lo = smem_desc_sw128(sb + oXG + T128 + ks * 32, 16, 1024);
            const uint64_t b_hi = smem_desc_sw128(sb + oX + ks * 16 * 128, C * 128, 1024);
            const uint64_t b_lo = smem_desc_sw128(sb + oX + 64 * 128 + ks * 16 * 128, C * 128, 1024);
            mma_bf16(tmem + G::T_D, a_hi, b_hi, id_x, ks > 0);
            mma_bf16(tmem + G::T_D, a_hi, b_lo, id_x, 1u);
            mma_bf16(tmem + G::T_D, a_lo, b_hi, id_x, 1u);
        }
        mma_commit(mbar);
    }
    if (ok) ok = mma_wait();
    // operands: X G (for W) and X (for U), K-major rows, from TMEM
    if (ok) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_off + G::T_D + cq * 16, v);
        tmem_ld_wait();
#pragma unroll
        for (int j8 = 0; j8 < 16; j8 += 8) {
            float xr[8], xg[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                xr[e] = __uint_as_float(v[j8 + e]);
                xg[e] = xr[e] * Gs[cq * 16 + j8 + e];
            }
            uint4 hi, lo;
            const uint32_t off = sw128_off16(row, cq * 16 + j8, 128);
            if (do_w) {
                split8(xg, hi, lo);
                V4(oXG + off) = hi;
                V4(oXG + T128 + off) = lo;
            }
            if (do_u) {
                split8(xr, hi, lo);
                V4(oX + off) = hi;
                V4(oX + T128 + off) = lo;
            }
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    // ---------------------------------------------------------------- [W | U] = X [G K | V]
    if (ok && tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks) {
            const uint64_t bk = smem_desc_sw128(sb + oKQ + ks * 2048, kq_region, 1024);
            const uint64_t bvv = smem_desc_sw128(sb + oV + ks * 2048, C * 128, 1024);
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {             // the hi and lo halves of the X operand
                const uint32_t ao = hl * T128 + ks * 32;
                if (do_w)
                    mma_bf16(tmem + G::T_WU, smem_desc_sw128(sb + oXG + ao, 16, 1024), bk,
                             idesc_bf16_f32(128, DK, true), (ks | hl) != 0);
                if (do_u)
                    mma_bf16(tmem + G::T_WU + DK, smem_desc_sw128(sb + oX + ao, 16, 1024), bvv,
                             idesc_bf16_f32(128, dv, true), (ks | hl) != 0);
            }
        }
        mma_commit(mbar);
    }
    if (ok) ok = mma_wait();
    // ---------------------------------------------------------------- v2 record
    // TMEM T_WU holds W (rows < 64) | A W (rows >= 64) in columns [0, DK) and
    // U | A U in [DK, DK + dv).  Thread (row, cq) takes 16-column pieces.
    //  (1) operands w W, w U (rows < 64, scaled by w_t) for P_c and B_c, and
    //      the record's Q' = G Q - A W (hi | lo) and A U (fp32) (rows >= 64)
    {
        const int t = row & 63;
        const float gt = Gs[t];
        const float wt = ws[t];
        float* au = reinterpret_cast<float*>(smem + G2::OFF_AU);
        for (int k = 0; k < DK / 64 && ok; ++k) {
            const int cb = 64 * k + 16 * cq;
            uint32_t v[16];
            tmem_ld16(tmem + lane_off + G::T_WU + cb, v);
            tmem_ld_wait();
            float y[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) y[j] = __uint_as_float(v[j]);
            if (row < 64) {
#pragma unroll
                for (int j = 0; j < 16; ++j) y[j] *= wt;
            } else {
#pragma unroll
                for (int j8 = 0; j8 < 16; j8 += 8) {
                    const uint4 q8 = V4(oKQ + sw128_off16(row, cb + j8, 128));
                    const uint32_t* qw = reinterpret_cast<const uint32_t*>(&q8);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 f2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&qw[e]));
                        y[j8 + 2 * e] = gt * f2.x - y[j8 + 2 * e];
                        y[j8 + 2 * e + 1] = gt * f2.y - y[j8 + 2 * e + 1];
                    }
                }
            }
            const uint32_t base = row < 64 ? G2::OFF_WW : G2::OFF_QI;
            const uint32_t halfb = row < 64 ? G2::WW_HALF : (uint32_t)R::QH;
#pragma unroll
            for (int j8 = 0; j8 < 16; j8 += 8) {
                uint4 hi, lo;
                split8(y + j8, hi, lo);
                const uint32_t off = sw128_off16(t, cb + j8, 64);
                V4(base + off) = hi;
                V4(base + halfb + off) = lo;
            }
        }
        for (int k = 0; k < (dv + 63) / 64 && ok; ++k) {
            const int rc = 64 * k + 16 * cq;
            if (rc >= dv) continue;                  // uniform per warp
            uint32_t v[16];
            tmem_ld16(tmem + lane_off + G::T_WU + DK + rc, v);
            tmem_ld_wait();
            if (row < 64) {
                float y[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) y[j] = __uint_as_float(v[j]) * wt;
#pragma unroll
                for (int j8 = 0; j8 < 16; j8 += 8) {
                    uint4 hi, lo;
                    split8(y + j8, hi, lo);
                    const uint32_t off = sw128_off16(t, rc + j8, 64);
                    V4(G2::OFF_WU + off) = hi;
                    V4(G2::OFF_WU + G2::WU_HALF + off) = lo;
                }
            } else {
#pragma unroll
                for (int j4 = 0; j4 < 16; j4 += 4)
                    *reinterpret_cast<uint4*>(au + au_idx(t, rc + j4)) = make_uint4(v[j4], v[j4 + 1], v[j4 + 2], v[j4 + 3]);
            }
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    //  (2) P' = K^T (w W) and B_c = K^T (w U) on the tensor cores (K^T as the
    //      MN-major view of the [K; Q] tile's first 64 rows); Q' and A U leave
    if (ok && tid == 0) {
        tc_fence_after();
        const uint32_t id_p = idesc_bf16_f32(128, DK, true, true);
        const uint32_t id_b = idesc_bf16_f32(128, dv, true, true);
#pragma unroll
        for (int ks = 0; ks < C / 16; ++ks) {
            const uint64_t a = smem_desc_sw128(sb + oKQ + ks * 2048, kq_region, 1024);
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                mma_bf16(tmem + G2::T_P, a, smem_desc_sw128(sb + G2::OFF_WW + hl * G2::WW_HALF + ks * 2048, 64 * 128, 1024),
                         id_p, (ks | hl) != 0);
                mma_bf16(tmem + G2::T_B, a, smem_desc_sw128(sb + G2::OFF_WU + hl * G2::WU_HALF + ks * 2048, 64 * 128, 1024),
                         id_b, (ks | hl) != 0);
            }
        }
        mma_commit(mbar);
        bulk_store(rec + R::qi_off(), sb + G2::OFF_QI, 2 * (uint32_t)R::QH);
        bulk_store(rec + R::au_off(dv), sb + G2::OFF_AU, 64 * dv * 4);
        bulk_commit();
    }
    if (ok) ok = mma_wait();
    if (tid == 0) bulk_wait_read();                  // the Q' and A U staging is read before B_c overwrites it
    __syncthreads();
    //  (3) P_c = G_C I - P' (hi | lo, the chain's K-major A operand, rows = d_k)
    //      and B_c (fp32, in 32-column slices) staged, then stored
    {
        const float gC = gC_sh;
        float* bc = reinterpret_cast<float*>(smem + G2::OFF_BC);
        for (int k = 0; k < DK / 64 && ok; ++k) {
            const int cb = 64 * k + 16 * cq;
            uint32_t v[16];
            tmem_ld16(tmem + lane_off + G2::T_P + cb, v);
            tmem_ld_wait();
            float y[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) y[j] = (cb + j == row ? gC : 0.f) - __uint_as_float(v[j]);
#pragma unroll
            for (int j8 = 0; j8 < 16; j8 += 8) {
                uint4 hi, lo;
                split8(y + j8, hi, lo);
                const uint32_t off = sw128_off16(row, cb + j8, 128);
                V4(G2::OFF_PI + off) = hi;
                V4(G2::OFF_PI + (uint32_t)R::WQH + off) = lo;
            }
        }
        for (int k = 0; k < (dv + 63) / 64 && ok; ++k) {
            const int rc = 64 * k + 16 * cq;
            if (rc >= dv) continue;                  // uniform per warp
            uint32_t v[16];
            tmem_ld16(tmem + lane_off + G2::T_B + rc, v);
            tmem_ld_wait();
#pragma unroll
            for (int j4 = 0; j4 < 16; j4 += 4)
                *reinterpret_cast<uint4*>(bc + uau_idx(row, rc + j4)) = make_uint4(v[j4], v[j4 + 1], v[j4 + 2], v[j4 + 3]);
        }
    }
    fence_proxy_async_smem();
    __syncthreads();
    if (ok && tid == 0) {
        bulk_store(rec + R::pi_off(), sb + G2::OFF_PI, 2 * (uint32_t)R::WQH);
        bulk_store(rec + R::bc_off(), sb + G2::OFF_BC, 128 * dv * 4);
        bulk_commit();
        bulk_wait_read();
    }
    tc_fence_before();
    __syncthreads();                                 // the staging area is free for the next unit
    tc_fence_after();
    if (fc.flags && tid == 0 && ok) {
        bulk_wait_all();
        fence_proxy_async_global();
        __threadfence();
        st_release_u32(fc.flags + (int64_t)ch_h * kFlagWords, fc.epoch);
    }
    }  // units
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(*tmem_slot, 512);
    }
}

template <int DK>
__global__ void __launch_bounds__(kPrepThreads, 1) gdn_prep2_kernel(const __grid_constant__ GdnParams p) {
    gdn_prep2_run<DK>(p, FuseCtl{nullptr, 0}, blockIdx.x, gridDim.x);
}

// ============================================================================
// scan: one block per (character, head, d_v slice), chunks in order
// ============================================================================
template <int DK>
struct ScanCfg {
    static constexpr int WQ = 2 * (int)Rec<DK>::WQH;         // [W;Q'] hi | lo image
    static constexpr int KI = (int)Rec<DK>::KIMG;            // K image
    static constexpr int UAU = 128 * DVP * 4;                // U | A U (whole record row width dv <= 256)
    static constexpr int SOP = 2 * DK * DVMAX * 2;           // S hi, lo (rows c); w E hi, lo aliased
    static constexpr int OFF_WQ = 0;
    static constexpr int OFF_K = OFF_WQ + WQ;
    static constexpr int OFF_U = OFF_K + KI;
    static constexpr int OFF_S = OFF_U + UAU / 2;            // U | A U is staged for dv <= 128 (64 KB)
    static constexpr int OFF_BAR = OFF_S + SOP;
    static constexpr int SMEM = OFF_BAR + 64 + 1024;
    static constexpr uint32_t T_D = 0;                       // [W;Q'] S0^T (dv cols)
    static constexpr uint32_t T_S = 128;                     // S^T (dv cols)
};

// CW: columns of the slice a thread handles per TMEM access (16 when the
// slice is 32 wide, so that all eight warps share the elementwise phases)
// One scan item: character b, head h, d_v rows r0 .. r0 + dv_slice - 1.
// Written for 256 threads (eight warps: lane quarter x column half); in a
// fused launch's 512-thread blocks the other eight warps only take part in
// the block barriers (their column range is empty).
template <int DK, int CW>
__device__ __forceinline__ void gdn_scan_run(const GdnParams& p, const FuseCtl& fc, int b, int h, int r0) {
    using G = ScanCfg<DK>;
    using R = Rec<DK>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oS = G::OFF_S;
    constexpr uint32_t SH = DK * DVMAX * 2;                      // one S half
    constexpr uint32_t WEH = C * DVMAX * 2;                      // one w E half
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 32);
    const uint32_t mbar = smem_u32(&bars[0]);
    const uint32_t bar_wq = smem_u32(&bars[1]), bar_k = smem_u32(&bars[2]), bar_u = smem_u32(&bars[3]);
    const float* Us = reinterpret_cast<const float*>(smem + G::OFF_U);
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, hf = warp >> 2;
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int dvs = p.dv_slice;
    const GdnChar ch = p.ch[b];
    if (ch.M <= 0) return;                           // uniform per block; touches no memory
    const int H = p.H, dv = p.dv;
    const int nch = (ch.M + C - 1) / C;
    const uint32_t ubytes = 128u * dvs * 4u;         // the block's slice of U | A U
    const int64_t uslice = R::uau_off() + (int64_t)r0 * 128 * 4;
    float* Sg = p.S + ((int64_t)b * H + h) * dv * DK;
    const int dhalf = ((dvs / 2) + CW - 1) / CW * CW;
    const int dlo = hf * dhalf, dhi = min(dvs, dlo + dhalf);
    auto rec_of = [&](int i) -> const uint8_t* { return p.work + ((int64_t)(ch.chunk_off + i) * H + h) * p.rec_bytes; };

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        mbar_init(bar_wq, 1);
        mbar_init(bar_k, 1);
        mbar_init(bar_u, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    auto write_s_row = [&](int c, int rc, const float* x) {
#pragma unroll
        for (int j8 = 0; j8 < CW; j8 += 8) {
            if (rc + j8 < dvs) {
                uint4 hi, lo;
                split8(x + j8, hi, lo);
                const uint32_t off = sw128_off16(c, rc + j8, DK);
                V4(oS + off) = hi;
                V4(oS + SH + off) = lo;
            }
        }
    };
    // ---- the state slice: S^T into TMEM (lane c, column r) and the MN-major operand
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const int rc = dlo + CW * half;
        if (rc >= dhi) continue;                     // uniform per warp
        float sx[CW];
#pragma unroll
        for (int j = 0; j < CW; ++j)                 // all loads before any use
            sx[j] = (row < DK && rc + j < dhi) ? Sg[(int64_t)(r0 + rc + j) * DK + row] : 0.f;
        uint32_t v[CW];
#pragma unroll
        for (int j = 0; j < CW; ++j) v[j] = __float_as_uint(sx[j]);
        tmem_stw<CW>(tmem + lane_off + G::T_S + rc, v);
        if (row < DK) write_s_row(row, rc, sx);
    }
    tmem_st_wait();
    // The state slice comes from an earlier round (or kvm_set_state), which
    // completed before the prep kernel this launch follows had started, so
    // it is staged before waiting for that kernel; its records are not.
    if (!fc.flags) {                                 // the fused kernel waited already
        grid_dependency_wait();
        grid_dependents_launch();
    }
    // fused: the first record must have been published (a failed wait
    // raises the abort flag, which stops the block at its first MMA wait)
    if (tid == 0 && wait_record(fc, (int64_t)ch.chunk_off * H + h, &abort_flag, p.err, p.diag, 0x5f)) {
        mbar_arrive_expect_tx(bar_wq, G::WQ);
        bulk_load(sb + G::OFF_WQ, rec_of(0), G::WQ, bar_wq);
        mbar_arrive_expect_tx(bar_k, G::KI);
        bulk_load(sb + G::OFF_K, rec_of(0) + G::WQ, G::KI, bar_k);
        mbar_arrive_expect_tx(bar_u, ubytes);
        bulk_load(sb + G::OFF_U, rec_of(0) + uslice, ubytes, bar_u);
    }

    uint32_t phase = 0;
    bool ok = true;
    // the issuing thread waits for its MMAs and the block follows it at the
    // barrier (waiting lanes of the issuer's warp would slow its issue)
    auto mma_wait = [&]() -> bool {
        bool r = true;
        if (tid == 0) r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait, p.diag, 0x50);
        phase ^= 1;
        r = __syncthreads_and(r);
        tc_fence_after();
        return r;
    };
    auto issue_begin = [&]() { fence_proxy_async_smem(); tc_fence_before(); __syncthreads(); };
    const uint32_t id_1 = idesc_bf16_f32(128, dvs, true);           // B = S, MN-major
    const uint32_t id_2 = idesc_bf16_f32(128, dvs, true, true);     // A = K, B = w E, both MN-major
    const uint32_t kq_region = 128 * 128;
    issue_begin();

    for (int i = 0; i < nch && ok; ++i) {
        const int n = min(C, ch.M - i * C);
        const int64_t tok0 = ch.tail_off + (int64_t)i * C;
        const uint8_t* rec = rec_of(i);
        const float* misc = reinterpret_cast<const float*>(rec + R::misc_off(dv));
        // L2-coherent loads: in a fused launch the record was written by
        // another block of this grid
        const float wt = __ldcg(misc + (row & 63));
        const float gC = __ldcg(misc + C);
        // ---------------------------------------------------------------- [W; Q'] S0^T
        // Only the issuing thread reads the [W; Q'] image, so only it waits
        // for the copy; the state operand was published by the barrier that
        // ended the previous chunk.  A failed wait raises the abort flag,
        // which the MMA wait below turns into a block-wide stop.
        if (tid == 0 && mbar_wait(bar_wq, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x51 + 256 * i)) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t ao = (ks >> 2) * kq_region + (ks & 3) * 32;
                const uint32_t bo = ks * 2048;
                const uint64_t a_hi = smem_desc_sw128(sb + G::OFF_WQ + ao, 16, 1024);
                const uint64_t a_lo = smem_desc_sw128(sb + G::OFF_WQ + (uint32_t)R::WQH + ao, 16, 1024);
                const uint64_t b_hi = smem_desc_sw128(sb + oS + bo, DK * 128, 1024);
                const uint64_t b_lo = smem_desc_sw128(sb + oS + SH + bo, DK * 128, 1024);
                mma_bf16(tmem + G::T_D, a_hi, b_hi, id_1, ks > 0);
                mma_bf16(tmem + G::T_D, a_hi, b_lo, id_1, 1u);
                mma_bf16(tmem + G::T_D, a_lo, b_hi, id_1, 1u);
            }
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        // [W;Q'] image consumed: fetch the next one (fused: once the prep
        // has published that record; a failed wait raises the abort flag)
        if (tid == 0 && i + 1 < nch &&
            wait_record(fc, (int64_t)(ch.chunk_off + i + 1) * H + h, &abort_flag, p.err, p.diag, 0x5e + 256 * i)) {
            mbar_arrive_expect_tx(bar_wq, G::WQ);
            bulk_load(sb + G::OFF_WQ, rec_of(i + 1), G::WQ, bar_wq);
        }
        // ---------------------------------------------------------------- E, O; S^T *= G_C
        // every thread waits for the U | A U copy it reads; a failed wait
        // stops the block at the barrier after this phase
        const bool u_ok = mbar_wait(bar_u, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x52 + 256 * i);
        {
            const int t = row & 63;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const int rc = dlo + CW * half;
                if (rc >= dhi) continue;                 // uniform per warp
                uint32_t d1[CW], sv[CW];
                tmem_ldw<CW>(tmem + lane_off + G::T_D + rc, d1);
                tmem_ldw<CW>(tmem + lane_off + G::T_S + rc, sv);
                float u[CW];
#pragma unroll
                for (int j4 = 0; j4 < CW; j4 += 4) {
                    const float4 f = *reinterpret_cast<const float4*>(Us + uau_idx(row, rc + j4));
                    u[j4] = f.x; u[j4 + 1] = f.y; u[j4 + 2] = f.z; u[j4 + 3] = f.w;
                }
                tmem_ld_wait();
                if (row < 64) {
                    float e[CW];
#pragma unroll
                    for (int j = 0; j < CW; ++j) e[j] = wt * (u[j] - __uint_as_float(d1[j]));
#pragma unroll
                    for (int j8 = 0; j8 < CW; j8 += 8) {
                        if (rc + j8 < dvs) {
                            uint4 hi, lo;
                            split8(e + j8, hi, lo);
                            const uint32_t off = sw128_off16(t, rc + j8, C);
                            V4(oS + off) = hi;                  // w E aliases the S operand
                            V4(oS + WEH + off) = lo;
                        }
                    }
                } else if (t < n) {
                    __nv_bfloat16* o = p.out + ((tok0 + t) * H + h) * dv + r0 + rc;
#pragma unroll
                    for (int j8 = 0; j8 < CW; j8 += 8) {
                        if (rc + j8 < dvs) {
                            uint4 w4;
                            uint32_t* ww = reinterpret_cast<uint32_t*>(&w4);
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                ww[e] = pack_bf16x2(u[j8 + 2 * e] + __uint_as_float(d1[j8 + 2 * e]),
                                                    u[j8 + 2 * e + 1] + __uint_as_float(d1[j8 + 2 * e + 1]));
                            *reinterpret_cast<uint4*>(o + j8) = w4;
                        }
                    }
                }
#pragma unroll
                for (int j = 0; j < CW; ++j) sv[j] = __float_as_uint(__uint_as_float(sv[j]) * gC);
                tmem_stw<CW>(tmem + lane_off + G::T_S + rc, sv);
            }
            tmem_st_wait();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        ok = __syncthreads_and(u_ok);
        if (!ok) break;
        if (tid == 0 && i + 1 < nch && !abort_flag) {   // U | A U consumed: fetch the next one
            mbar_arrive_expect_tx(bar_u, ubytes);
            bulk_load(sb + G::OFF_U, rec_of(i + 1) + uslice, ubytes, bar_u);
        }
        // ---------------------------------------------------------------- S^T += K^T (w E)
        // only the issuing thread reads the K image
        if (tid == 0 && mbar_wait(bar_k, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x53 + 256 * i)) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < C / 16; ++ks) {
                const uint64_t a = smem_desc_sw128(sb + G::OFF_K + ks * 2048, C * 128, 1024);
                mma_bf16(tmem + G::T_S, a, smem_desc_sw128(sb + oS + ks * 2048, C * 128, 1024), id_2, 1u);
                mma_bf16(tmem + G::T_S, a, smem_desc_sw128(sb + oS + WEH + ks * 2048, C * 128, 1024), id_2, 1u);
            }
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        if (tid == 0 && i + 1 < nch && !abort_flag) {   // K image consumed: fetch the next one
            mbar_arrive_expect_tx(bar_k, G::KI);
            bulk_load(sb + G::OFF_K, rec_of(i + 1) + G::WQ, G::KI, bar_k);
        }
        // ---------------------------------------------------------------- refresh the state operand
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int rc = dlo + CW * half;
            if (rc >= dhi) continue;                     // uniform per warp
            uint32_t sv[CW];
            tmem_ldw<CW>(tmem + lane_off + G::T_S + rc, sv);
            tmem_ld_wait();
            if (row < DK) {
                float y[CW];
#pragma unroll
                for (int j = 0; j < CW; ++j) y[j] = __uint_as_float(sv[j]);
                write_s_row(row, rc, y);
            }
        }
        issue_begin();
    }
    if (ok) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int rc = dlo + CW * half;
            if (rc >= dhi) continue;                     // uniform per warp
            uint32_t sv[CW];
            tmem_ldw<CW>(tmem + lane_off + G::T_S + rc, sv);
            tmem_ld_wait();
            if (row < DK) {
#pragma unroll
                for (int j = 0; j < CW; ++j)
                    if (rc + j < dvs) Sg[(int64_t)(r0 + rc + j) * DK + row] = __uint_as_float(sv[j]);
            }
        }
    } else if (tid == 0) {
        // let outstanding record copies land before the block exits
        volatile int never = 0;
        const uint32_t bs3[3] = {bar_wq, bar_k, bar_u};
        for (int k = 0; k < 3; ++k) {
            mbar_wait(bs3[k], 0, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
            mbar_wait(bs3[k], 1, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

// Scan of a slice of at most 32 d_v rows with hi | lo packed side by side in
// one 64-column operand.  The MMAs of the chain are short (N <= 64), so their
// cost is per instruction rather than per column: [W; Q'] (hi, then lo)
// against [S_hi | S_lo] takes 2 DK/16 MMAs instead of 3 DK/16, and
// K^T [wE_hi | wE_lo] takes C/16 instead of 2 C/16.  Each product's two
// halves land in columns c and 32 + c of its accumulator and are added when
// read.  The state stays fp32 in the threads' registers (thread (row,
// column half) holds S^T[row][16 columns]); TMEM holds only the two
// products:
//     D1 = [W; Q'] [S_hi | S_lo]             E = w (U - D1a - D1b),  O = A U + D1a + D1b
//     D2 = K^T [wE_hi | wE_lo]               S^T = G_C S^T + D2a + D2b
template <int DK>
__device__ __forceinline__ void gdn_scan_packed_run(const GdnParams& p, const FuseCtl& fc, int b, int h, int r0) {
    using G = ScanCfg<DK>;
    using R = Rec<DK>;
    constexpr int CW = 16;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oS = G::OFF_S;                // [S_hi | S_lo]: DK rows of 128 bytes; [wE_hi | wE_lo] (C rows) aliases it
    constexpr uint32_t T_D1 = 0, T_D2 = 128;         // 64 columns each
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 32);
    const uint32_t mbar = smem_u32(&bars[0]);
    const uint32_t bar_wq = smem_u32(&bars[1]), bar_k = smem_u32(&bars[2]), bar_u = smem_u32(&bars[3]);
    const float* Us = reinterpret_cast<const float*>(smem + G::OFF_U);
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, hf = warp >> 2;
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int dvs = p.dv_slice;                      // <= 32
    const GdnChar ch = p.ch[b];
    if (ch.M <= 0) return;                           // uniform per block; touches no memory
    // The scan runs on warps 0-7 and synchronises them with barrier 1 of 256
    // threads; the other warps of a fused launch's 512-thread block leave.
    if (warp >= kThreads / 32) return;
    auto sync = [&]() { named_bar_sync(1, kThreads); };
    auto sync_and = [&](bool x) { return named_bar_and(1, kThreads, x); };
    const int H = p.H, dv = p.dv;
    const int nch = (ch.M + C - 1) / C;
    const uint32_t ubytes = 128u * dvs * 4u;
    const int64_t uslice = R::uau_off() + (int64_t)r0 * 128 * 4;
    float* Sg = p.S + ((int64_t)b * H + h) * dv * DK;
    const int rc = hf * CW;                          // columns rc .. rc + 15 of the slice
    const bool cols = hf < 2 && rc < dvs;            // uniform per warp (fused blocks: warps 8.. have none)
    auto rec_of = [&](int i) -> const uint8_t* { return p.work + ((int64_t)(ch.chunk_off + i) * H + h) * p.rec_bytes; };

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        mbar_init(bar_wq, 1);
        mbar_init(bar_k, 1);
        mbar_init(bar_u, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 256);
        tmem_relinquish();
    }
    // columns no thread owns (slices narrower than 32) stay zero
    for (int i = tid; i < DK * 128 / 16; i += kThreads) V4(oS + 16 * i) = make_uint4(0, 0, 0, 0);
    tc_fence_before();
    sync();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // row `row` of S^T, hi at column c and lo at column 32 + c of the operand
    auto write_s = [&](int r, const float* x) {
#pragma unroll
        for (int j8 = 0; j8 < CW; j8 += 8) {
            if (rc + j8 < dvs) {
                uint4 hi, lo;
                split8(x + j8, hi, lo);
                V4(oS + sw128_off16(r, rc + j8, DK)) = hi;
                V4(oS + sw128_off16(r, 32 + rc + j8, DK)) = lo;
            }
        }
    };
    float sreg[CW];
#pragma unroll
    for (int j = 0; j < CW; ++j)                     // all loads before any use
        sreg[j] = (cols && row < DK && rc + j < dvs) ? Sg[(int64_t)(r0 + rc + j) * DK + row] : 0.f;
    if (cols && row < DK) write_s(row, sreg);
    // The state slice comes from an earlier round (or kvm_set_state), which
    // completed before the prep kernel this launch follows had started, so
    // it is staged before waiting for that kernel; its records are not.
    grid_dependency_wait();
    grid_dependents_launch();
    if (tid == 0 && wait_record(fc, (int64_t)ch.chunk_off * H + h, &abort_flag, p.err, p.diag, 0x5f)) {
        mbar_arrive_expect_tx(bar_wq, G::WQ);
        bulk_load(sb + G::OFF_WQ, rec_of(0), G::WQ, bar_wq);
        mbar_arrive_expect_tx(bar_k, G::KI);
        bulk_load(sb + G::OFF_K, rec_of(0) + G::WQ, G::KI, bar_k);
        mbar_arrive_expect_tx(bar_u, ubytes);
        bulk_load(sb + G::OFF_U, rec_of(0) + uslice, ubytes, bar_u);
    }

    uint32_t phase = 0;
    bool ok = true;
    auto mma_wait = [&]() -> bool {
        bool r = true;
        if (tid == 0) r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait, p.diag, 0x50);
        phase ^= 1;
        r = sync_and(r);
        tc_fence_after();
        return r;
    };
    auto issue_begin = [&]() { fence_proxy_async_smem(); tc_fence_before(); sync(); };
    const uint32_t id_1 = idesc_bf16_f32(128, 64, true);           // B = [S_hi | S_lo], MN-major
    const uint32_t id_2 = idesc_bf16_f32(128, 64, true, true);     // A = K, B = [wE_hi | wE_lo], both MN-major
    const uint32_t kq_region = 128 * 128;
    issue_begin();

    for (int i = 0; i < nch && ok; ++i) {
        const int n = min(C, ch.M - i * C);
        const int64_t tok0 = ch.tail_off + (int64_t)i * C;
        const uint8_t* rec = rec_of(i);
        const float* misc = reinterpret_cast<const float*>(rec + R::misc_off(dv));
        const float wt = __ldcg(misc + (row & 63));
        const float gC = __ldcg(misc + C);
        // ---------------------------------------------------------------- D1 = [W; Q'] [S_hi | S_lo]
        if (tid == 0 && mbar_wait(bar_wq, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x51 + 256 * i)) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t ao = (ks >> 2) * kq_region + (ks & 3) * 32;
                const uint64_t bs = smem_desc_sw128(sb + oS + ks * 2048, DK * 128, 1024);
                mma_bf16(tmem + T_D1, smem_desc_sw128(sb + G::OFF_WQ + ao, 16, 1024), bs, id_1, ks > 0);
                mma_bf16(tmem + T_D1, smem_desc_sw128(sb + G::OFF_WQ + (uint32_t)R::WQH + ao, 16, 1024), bs, id_1, 1u);
            }
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        if (tid == 0 && i + 1 < nch &&
            wait_record(fc, (int64_t)(ch.chunk_off + i + 1) * H + h, &abort_flag, p.err, p.diag, 0x5e + 256 * i)) {
            mbar_arrive_expect_tx(bar_wq, G::WQ);
            bulk_load(sb + G::OFF_WQ, rec_of(i + 1), G::WQ, bar_wq);
        }
        // ---------------------------------------------------------------- E (rows < 64) and O (rows >= 64)
        const bool u_ok = !cols || mbar_wait(bar_u, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x52 + 256 * i);
        if (cols) {
            const int t = row & 63;
            uint32_t da[CW], db[CW];
            tmem_ldw<CW>(tmem + lane_off + T_D1 + rc, da);
            tmem_ldw<CW>(tmem + lane_off + T_D1 + 32 + rc, db);
            float u[CW];
#pragma unroll
            for (int j4 = 0; j4 < CW; j4 += 4) {
                const float4 f = *reinterpret_cast<const float4*>(Us + uau_idx(row, rc + j4));
                u[j4] = f.x; u[j4 + 1] = f.y; u[j4 + 2] = f.z; u[j4 + 3] = f.w;
            }
            tmem_ld_wait();
            float d[CW];
#pragma unroll
            for (int j = 0; j < CW; ++j) d[j] = __uint_as_float(da[j]) + __uint_as_float(db[j]);
            if (row < 64) {
                float e[CW];
#pragma unroll
                for (int j = 0; j < CW; ++j) e[j] = wt * (u[j] - d[j]);
#pragma unroll
                for (int j8 = 0; j8 < CW; j8 += 8) {
                    if (rc + j8 < dvs) {
                        uint4 hi, lo;
                        split8(e + j8, hi, lo);
                        V4(oS + sw128_off16(t, rc + j8, C)) = hi;          // [wE_hi | wE_lo] aliases the S operand
                        V4(oS + sw128_off16(t, 32 + rc + j8, C)) = lo;
                    }
                }
            } else if (t < n) {
                __nv_bfloat16* o = p.out + ((tok0 + t) * H + h) * dv + r0 + rc;
#pragma unroll
                for (int j8 = 0; j8 < CW; j8 += 8) {
                    if (rc + j8 < dvs) {
                        uint4 w4;
                        uint32_t* ww = reinterpret_cast<uint32_t*>(&w4);
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            ww[e] = pack_bf16x2(u[j8 + 2 * e] + d[j8 + 2 * e], u[j8 + 2 * e + 1] + d[j8 + 2 * e + 1]);
                        *reinterpret_cast<uint4*>(o + j8) = w4;
                    }
                }
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        ok = sync_and(u_ok);
        if (!ok) break;
        if (tid == 0 && i + 1 < nch && !abort_flag) {
            mbar_arrive_expect_tx(bar_u, ubytes);
            bulk_load(sb + G::OFF_U, rec_of(i + 1) + uslice, ubytes, bar_u);
        }
        // ---------------------------------------------------------------- D2 = K^T [wE_hi | wE_lo]
        if (tid == 0 && mbar_wait(bar_k, i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x53 + 256 * i)) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < C / 16; ++ks)
                mma_bf16(tmem + T_D2, smem_desc_sw128(sb + G::OFF_K + ks * 2048, C * 128, 1024),
                         smem_desc_sw128(sb + oS + ks * 2048, C * 128, 1024), id_2, ks > 0);
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        if (tid == 0 && i + 1 < nch && !abort_flag) {
            mbar_arrive_expect_tx(bar_k, G::KI);
            bulk_load(sb + G::OFF_K, rec_of(i + 1) + G::WQ, G::KI, bar_k);
        }
        // ---------------------------------------------------------------- S^T = G_C S^T + D2a + D2b
        if (cols) {
            uint32_t da[CW], db[CW];
            tmem_ldw<CW>(tmem + lane_off + T_D2 + rc, da);
            tmem_ldw<CW>(tmem + lane_off + T_D2 + 32 + rc, db);
            tmem_ld_wait();
            if (row < DK) {
#pragma unroll
                for (int j = 0; j < CW; ++j) sreg[j] = fmaf(gC, sreg[j], __uint_as_float(da[j]) + __uint_as_float(db[j]));
                write_s(row, sreg);
            }
        }
        issue_begin();
    }
    if (ok) {
        if (cols && row < DK) {
#pragma unroll
            for (int j = 0; j < CW; ++j)
                if (rc + j < dvs) Sg[(int64_t)(r0 + rc + j) * DK + row] = sreg[j];
        }
    } else if (tid == 0) {
        // let outstanding record copies land before the block exits
        volatile int never = 0;
        const uint32_t bs3[3] = {bar_wq, bar_k, bar_u};
        for (int k = 0; k < 3; ++k) {
            mbar_wait(bs3[k], 0, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
            mbar_wait(bs3[k], 1, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
        }
    }
    tc_fence_before();
    sync();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

template <int DK, int CW>
__global__ void __launch_bounds__(kThreads, 1) gdn_scan_kernel(const __grid_constant__ GdnParams p) {
    if constexpr (CW == 16) gdn_scan_packed_run<DK>(p, FuseCtl{nullptr, 0}, blockIdx.z, blockIdx.y, blockIdx.x * p.dv_slice);
    else gdn_scan_run<DK, CW>(p, FuseCtl{nullptr, 0}, blockIdx.z, blockIdx.y, blockIdx.x * p.dv_slice);
}

// ============================================================================
// fused: prep and scan in one launch.  Blocks 0 .. n_scan-1 each run one scan
// item (character, head, d_v slice); the others are prep workers that take
// the (chunk, head) units in fused_unit order and publish each record through
// its flag.  A scan waits only for records, and prep workers never wait, so
// the launch completes as long as every prep worker eventually gets an SM:
// the scan items leave at least kMinPrepWorkers SMs, other kernels' blocks
// (the compaction beside it) finish on their own, and the kernels after it
// on the stream cannot take an SM before every block of it has started
// (their launch waits for every block's launch_dependents).  Not a
// cooperative launch: that one waited for every SM to be free, and so for
// the compaction blocks beside it (a round 6.56 against 6.46 ms).
// ============================================================================
template <int DK, int CW>
__global__ void __launch_bounds__(kPrepThreads, 1) gdn_fused_kernel(const __grid_constant__ GdnParams p) {
    // each role waits for the previous grid after its own set-up (below)
    const FuseCtl fc{p.flags, p.epoch};
    const int x = blockIdx.x;
    if (x < p.n_scan) {
        const int slices = p.dv / p.dv_slice;
        gdn_scan_packed_run<DK>(p, fc, x / (slices * p.H), (x / slices) % p.H, (x % slices) * p.dv_slice);
    } else {
        gdn_prep_run<DK>(p, fc, x - p.n_scan, gridDim.x - p.n_scan);
    }
}

// ============================================================================
// v2 chain: one block per (character, head, d_v slice of 32 rows), chunks in
// order.  The state slice S^T (lane = d_k row, 32 columns) lives in the
// threads' registers in fp32 (thread (row, column half) holds 16 values) and,
// split hi | lo, in shared memory as the MN-major operand of the next MMA.
// Per chunk: D = P_c S0^T (24 MMAs), then S^T = D + B_c, the operand
// refreshed and the entering state of the next chunk written as its snapshot.
// P_c and the B_c slice of the next two chunks are in flight (two buffers).
// ============================================================================
template <int DK>
struct Chain2Cfg {
    using R = Rec2<DK>;
    static constexpr int DVS = 32;                           // d_v rows per block
    static constexpr int PI = 2 * (int)R::WQH;               // P_c hi | lo image
    static constexpr int BCS = 128 * DVS * 4;                // the block's B_c slice
    static constexpr int SOP = 2 * DK * 64 * 2;              // S hi, lo (one 64-column region each)
    static constexpr int OFF_PI = 0;                          // two buffers
    static constexpr int OFF_BC = OFF_PI + 2 * PI;            // two buffers
    static constexpr int OFF_S = OFF_BC + 2 * BCS;
    static constexpr int OFF_BAR = OFF_S + SOP;
    static constexpr int SMEM = OFF_BAR + 64 + 1024;
    static constexpr uint32_t T_D = 0;                        // P_c S0^T (DVS columns)
};

// Snapshot of the state entering chunk `chunk` of head h: the MN-major
// operand image [d_k][d_v] hi, then lo (each DK x d_v bf16 in 64-column
// regions), as the output kernel reads it.
__device__ __forceinline__ uint8_t* snap_of(const GdnParams& p, int64_t chunk, int h) {
    return p.snap + (chunk * p.H + h) * p.snap_bytes;
}

template <int DK>
__device__ __forceinline__ void gdn_chain2_run(const GdnParams& p, const FuseCtl& fc, int b, int h, int r0) {
    using G = Chain2Cfg<DK>;
    using R = Rec2<DK>;
    constexpr int CW = 16;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oS = G::OFF_S;
    constexpr uint32_t SH = DK * 64 * 2;                     // one S half
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 48);
    const uint32_t mbar = smem_u32(&bars[0]);
    const uint32_t bar_pi[2] = {smem_u32(&bars[1]), smem_u32(&bars[2])};
    const uint32_t bar_bc[2] = {smem_u32(&bars[3]), smem_u32(&bars[4])};
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, hf = warp >> 2;             // hf >= 2 (fused 512-thread blocks): no columns
    const int row = q4 * 32 + lane;                      // d_k row (TMEM lane)
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const GdnChar ch = p.ch[b];
    if (ch.M <= 0) return;                               // uniform per block; touches no memory
    const int H = p.H, dv = p.dv;
    const int nch = (ch.M + C - 1) / C;
    const int rc = hf * CW;                              // this thread's 16 columns of the slice
    const bool cols = hf < 2;
    float* Sg = p.S + ((int64_t)b * H + h) * dv * DK;
    auto rec_of = [&](int i) -> const uint8_t* { return p.work + ((int64_t)(ch.chunk_off + i) * H + h) * p.rec_bytes; };
    const int64_t bc_slice = R::bc_off() + (int64_t)r0 * 128 * 4;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        for (int k = 0; k < 2; ++k) {
            mbar_init(bar_pi[k], 1);
            mbar_init(bar_bc[k], 1);
        }
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 64);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // the state's operand image (this slice's columns of region 0) and its
    // snapshot (the slice's columns r0 .. r0 + 31 of the full-width image)
    auto put_state = [&](const float* x, int64_t snap_chunk) {
        uint8_t* snap = snap_of(p, snap_chunk, h);
#pragma unroll
        for (int j8 = 0; j8 < CW; j8 += 8) {
            uint4 hi, lo;
            split8(x + j8, hi, lo);
            const uint32_t off = sw128_off16(row, rc + j8, DK);
            V4(oS + off) = hi;
            V4(oS + SH + off) = lo;
            const uint32_t goff = sw128_off16(row, r0 + rc + j8, DK);
            *reinterpret_cast<uint4*>(snap + goff) = hi;
            *reinterpret_cast<uint4*>(snap + p.snap_bytes / 2 + goff) = lo;
        }
    };
    float st[CW];                                       // the master state (fp32)
    if (cols) {
#pragma unroll
        for (int j = 0; j < CW; ++j) st[j] = Sg[(int64_t)(r0 + rc + j) * DK + row];
    }
    if (!fc.flags) {                                     // the fused kernel waited already
        grid_dependency_wait();
        grid_dependents_launch();
    }
    if (cols) put_state(st, ch.chunk_off);
    // records of chunks 0 and 1
    if (tid == 0) {
        for (int i = 0; i < 2 && i < nch; ++i) {
            if (!wait_record(fc, (int64_t)(ch.chunk_off + i) * H + h, &abort_flag, p.err, p.diag, 0x6f)) break;
            mbar_arrive_expect_tx(bar_pi[i], G::PI);
            bulk_load(sb + G::OFF_PI + i * G::PI, rec_of(i) + R::pi_off(), G::PI, bar_pi[i]);
            mbar_arrive_expect_tx(bar_bc[i], G::BCS);
            bulk_load(sb + G::OFF_BC + i * G::BCS, rec_of(i) + bc_slice, G::BCS, bar_bc[i]);
        }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();

    uint32_t phase = 0;
    bool ok = true;
    const uint32_t id_c = idesc_bf16_f32(128, G::DVS, true);        // B = S, MN-major
    const uint32_t kq_region = 128 * 128;
    for (int i = 0; i < nch && ok; ++i) {
        const int buf = i & 1;
        const uint32_t par = (i >> 1) & 1;
        // ---------------------------------------------------------------- D = P_c S0^T
        if (tid == 0 && mbar_wait(bar_pi[buf], par, &abort_flag, p.err, kErrWait, p.diag, 0x61 + 256 * i)) {
            tc_fence_after();
            const uint32_t pb = sb + G::OFF_PI + buf * G::PI;
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t ao = (ks >> 2) * kq_region + (ks & 3) * 32;
                const uint64_t a_hi = smem_desc_sw128(pb + ao, 16, 1024);
                const uint64_t a_lo = smem_desc_sw128(pb + (uint32_t)R::WQH + ao, 16, 1024);
                const uint64_t b_hi = smem_desc_sw128(sb + oS + ks * 2048, DK * 128, 1024);
                const uint64_t b_lo = smem_desc_sw128(sb + oS + SH + ks * 2048, DK * 128, 1024);
                mma_bf16(tmem + G::T_D, a_hi, b_hi, id_c, ks > 0);
                mma_bf16(tmem + G::T_D, a_hi, b_lo, id_c, 1u);
                mma_bf16(tmem + G::T_D, a_lo, b_hi, id_c, 1u);
            }
            mma_commit(mbar);
        }
        // B_c of this chunk into registers while the MMAs run
        float bcv[CW];
        const bool bc_ok = mbar_wait(bar_bc[buf], par, &abort_flag, p.err, kErrWait, p.diag, 0x62 + 256 * i);
        if (cols) {
            const float* bc = reinterpret_cast<const float*>(smem + G::OFF_BC + buf * G::BCS);
#pragma unroll
            for (int j4 = 0; j4 < CW; j4 += 4) {
                const float4 f = *reinterpret_cast<const float4*>(bc + uau_idx(row, rc + j4));
                bcv[j4] = f.x; bcv[j4 + 1] = f.y; bcv[j4 + 2] = f.z; bcv[j4 + 3] = f.w;
            }
        }
        bool r = true;
        if (tid == 0) r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait, p.diag, 0x60);
        phase ^= 1;
        ok = __syncthreads_and(r && bc_ok);
        tc_fence_after();
        if (!ok) break;
        // ---------------------------------------------------------------- S^T = D + B_c, operand and snapshot
        if (cols) {
            uint32_t d[CW];
            tmem_ldw<CW>(tmem + lane_off + G::T_D + rc, d);
            tmem_ld_wait();
#pragma unroll
            for (int j = 0; j < CW; ++j) st[j] = __uint_as_float(d[j]) + bcv[j];
            if (i + 1 < nch) put_state(st, ch.chunk_off + i + 1);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        // the buffers of chunk i are consumed: fetch chunk i + 2 into them
        if (tid == 0 && i + 2 < nch &&
            wait_record(fc, (int64_t)(ch.chunk_off + i + 2) * H + h, &abort_flag, p.err, p.diag, 0x6e + 256 * i)) {
            mbar_arrive_expect_tx(bar_pi[buf], G::PI);
            bulk_load(sb + G::OFF_PI + buf * G::PI, rec_of(i + 2) + R::pi_off(), G::PI, bar_pi[buf]);
            mbar_arrive_expect_tx(bar_bc[buf], G::BCS);
            bulk_load(sb + G::OFF_BC + buf * G::BCS, rec_of(i + 2) + bc_slice, G::BCS, bar_bc[buf]);
        }
    }
    if (ok) {
        if (cols) {
#pragma unroll
            for (int j = 0; j < CW; ++j) Sg[(int64_t)(r0 + rc + j) * DK + row] = st[j];
        }
    } else if (tid == 0) {
        // let outstanding record copies land before the block exits
        volatile int never = 0;
        for (int k = 0; k < 2; ++k) {
            for (int q = 0; q < 2; ++q) {
                mbar_wait(bar_pi[k], q, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
                mbar_wait(bar_bc[k], q, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 64);
    }
}

template <int DK>
__global__ void __launch_bounds__(kThreads, 1) gdn_chain2_kernel(const __grid_constant__ GdnParams p) {
    gdn_chain2_run<DK>(p, FuseCtl{nullptr, 0}, blockIdx.z, blockIdx.y, blockIdx.x * 32);
}

// v2 fused: prep workers (gdn_prep2_run) and chain blocks in one grid, as
// gdn_fused_kernel.
template <int DK>
__global__ void __launch_bounds__(kPrepThreads, 1) gdn_fused2_kernel(const __grid_constant__ GdnParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const FuseCtl fc{p.flags, p.epoch};
    const int x = blockIdx.x;
    if (x < p.n_scan) {
        const int slices = p.dv / 32;
        gdn_chain2_run<DK>(p, fc, x / (slices * p.H), (x / slices) % p.H, (x % slices) * 32);
    } else {
        gdn_prep2_run<DK>(p, fc, x - p.n_scan, gridDim.x - p.n_scan);
    }
}

// ============================================================================
// v2 outputs: one block per (chunk, head): O = A U + Q' S0^T, with S0^T the
// chunk's snapshot.  Q' fills rows 0..63 of an M = 128 operand (rows 64..127
// zero); D rows 0..63 are the chunk's tokens.
// ============================================================================
template <int DK>
struct Out2Cfg {
    using R = Rec2<DK>;
    static constexpr int AI = 2 * 128 * DK * 2;              // Q' hi | lo as 128-row images
    static constexpr int OFF_A = 0;
    static constexpr int OFF_B = OFF_A + AI;                  // snapshot hi | lo (d_v <= 128)
    static constexpr int OFF_AU = OFF_B + 2 * DK * 128 * 2;
    static constexpr int OFF_BAR = OFF_AU + 64 * 128 * 4;
    static constexpr int SMEM = OFF_BAR + 64 + 1024;
};

template <int DK>
__global__ void __launch_bounds__(kThreads, 1) gdn_out2_kernel(const __grid_constant__ GdnParams p) {
    using G = Out2Cfg<DK>;
    using R = Rec2<DK>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 16);
    const uint32_t mbar = smem_u32(&bars[0]), bar_in = smem_u32(&bars[1]);
    __shared__ volatile int abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, hf = warp >> 2;
    const int row = q4 * 32 + lane;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int H = p.H, dv = p.dv;
    const int chunk = blockIdx.x / H, h = blockIdx.x % H;
    const int b = find_char_by_chunk(p, chunk);
    const GdnChar ch = p.ch[b];
    const int c0 = (chunk - ch.chunk_off) * C;
    if (c0 >= ch.M) return;                             // uniform per block (not reached for valid grids)
    const int n = min(C, ch.M - c0);
    const int64_t tok0 = ch.tail_off + c0;
    const uint8_t* rec = p.work + ((int64_t)chunk * H + h) * p.rec_bytes;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        mbar_init(bar_in, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 128);
        tmem_relinquish();
    }
    // rows 64..127 of the Q' operand are zero
    for (int idx = tid; idx < 2 * (DK / 64) * 64 * 8; idx += blockDim.x) {
        const int e = idx % 8, r64 = (idx / 8) % 64, rg = idx / 512;   // rg = half * regions + region
        *reinterpret_cast<uint4*>(smem + G::OFF_A + rg * (128 * 128) + (64 + r64) * 128 + e * 16) = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    grid_dependency_wait();
    grid_dependents_launch();
    if (tid == 0) {
        const uint32_t in_bytes = 2 * (uint32_t)R::QH + 2 * DK * dv * 2 + 64 * dv * 4;
        mbar_arrive_expect_tx(bar_in, in_bytes);
        for (int hl = 0; hl < 2; ++hl)
            for (int rg = 0; rg < DK / 64; ++rg)           // a 64-row region into rows 0..63 of a 128-row one
                bulk_load(sb + G::OFF_A + (hl * (DK / 64) + rg) * (128 * 128), rec + R::qi_off() + hl * R::QH + rg * (64 * 128),
                          64 * 128, bar_in);
        bulk_load(sb + G::OFF_B, snap_of(p, chunk, h), 2 * DK * dv * 2, bar_in);
        bulk_load(sb + G::OFF_AU, rec + R::au_off(dv), 64 * dv * 4, bar_in);
    }
    bool ok = true;
    if (tid == 0) {
        ok = mbar_wait(bar_in, 0, &abort_flag, p.err, kErrWait, p.diag, 0x71);
        if (ok) {
            tc_fence_after();
            const uint32_t id_o = idesc_bf16_f32(128, dv, true);      // B = snapshot, MN-major
            const uint32_t bhalf = DK * dv * 2;
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t ao = (ks >> 2) * (128 * 128) + (ks & 3) * 32;
                const uint64_t a_hi = smem_desc_sw128(sb + G::OFF_A + ao, 16, 1024);
                const uint64_t a_lo = smem_desc_sw128(sb + G::OFF_A + (DK / 64) * (128 * 128) + ao, 16, 1024);
                const uint64_t b_hi = smem_desc_sw128(sb + G::OFF_B + ks * 2048, DK * 128, 1024);
                const uint64_t b_lo = smem_desc_sw128(sb + G::OFF_B + bhalf + ks * 2048, DK * 128, 1024);
                mma_bf16(tmem, a_hi, b_hi, id_o, ks > 0);
                mma_bf16(tmem, a_hi, b_lo, id_o, 1u);
                mma_bf16(tmem, a_lo, b_hi, id_o, 1u);
            }
            mma_commit(mbar);
            ok = mbar_wait(mbar, 0, &abort_flag, p.err, kErrWait, p.diag, 0x72);
        }
    }
    ok = __syncthreads_and(ok);
    tc_fence_after();
    // rows 0..63 (warps with q4 < 2): O = A U + D, 16 columns at a time
    if (ok && q4 < 2) {
        const float* au = reinterpret_cast<const float*>(smem + G::OFF_AU);
        const int t = row;
        for (int c16 = hf * 16; c16 < dv; c16 += 32) {
            uint32_t d[16];
            tmem_ld16(tmem + lane_off + c16, d);
            tmem_ld_wait();
            if (t < n) {
                uint32_t w[8];
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    w[e] = pack_bf16x2(au[au_idx(t, c16 + 2 * e)] + __uint_as_float(d[2 * e]),
                                       au[au_idx(t, c16 + 2 * e + 1)] + __uint_as_float(d[2 * e + 1]));
                uint4* o = reinterpret_cast<uint4*>(p.out + ((tok0 + t) * H + h) * dv + c16);
                o[0] = make_uint4(w[0], w[1], w[2], w[3]);
                o[1] = make_uint4(w[4], w[5], w[6], w[7]);
            }
        }
    }
    if (!ok && tid == 0) {
        volatile int never = 0;
        mbar_wait(bar_in, 0, &never, p.err, kErrWait, nullptr, 0, 20000000ull);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 128);
    }
}

// Opt in to the kernel's dynamic shared memory once per device (one flag per
// kernel: the template is keyed on the kernel itself).
template <auto KERNEL>
void configure_once(int smem) {
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(KERNEL, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        configured |= 1ull << (dev & 63);
    }
}

template <int DK>
void launch_prep_dk(const GdnParams& p, cudaStream_t s) {
    configure_once<gdn_prep_kernel<DK>>(PrepCfg<DK>::SMEM);
    launch_pdl(gdn_prep_kernel<DK>, dim3(p.total_chunks * p.H * p.prep_parts), dim3(kPrepThreads), PrepCfg<DK>::SMEM, s, p);
}

template <int DK, int CW>
void launch_scan_cw(const GdnParams& p, cudaStream_t s) {
    configure_once<gdn_scan_kernel<DK, CW>>(ScanCfg<DK>::SMEM);
    dim3 grid(p.dv / p.dv_slice, p.H, p.n_chars);
    launch_pdl(gdn_scan_kernel<DK, CW>, grid, dim3(kThreads), ScanCfg<DK>::SMEM, s, p);
}

template <int DK>
void launch_scan_dk(const GdnParams& p, cudaStream_t s) {
    if (p.dv_slice <= 32) launch_scan_cw<DK, 16>(p, s);
    else launch_scan_cw<DK, 32>(p, s);
}

template <int DK>
cudaError_t launch_fused_dk(const GdnParams& p, int grid, cudaStream_t s) {
    constexpr int smem = ScanCfg<DK>::SMEM > PrepCfg<DK>::SMEM ? ScanCfg<DK>::SMEM : PrepCfg<DK>::SMEM;
    configure_once<gdn_fused_kernel<DK, 16>>(smem);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kPrepThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gdn_fused_kernel<DK, 16>, p);
}

template <int DK>
void launch_v2_dk(const GdnParams& p, int fused_grid, cudaStream_t s, cudaError_t* fused_err) {
    constexpr int fsmem = Chain2Cfg<DK>::SMEM > PrepCfg<DK>::SMEM ? Chain2Cfg<DK>::SMEM : PrepCfg<DK>::SMEM;
    if (fused_grid > 0) {
        configure_once<gdn_fused2_kernel<DK>>(fsmem);
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(fused_grid);
        cfg.blockDim = dim3(kPrepThreads);
        cfg.dynamicSmemBytes = fsmem;
        cfg.stream = s;
        cudaLaunchAttribute at[2];
        at[0].id = cudaLaunchAttributeCooperative;
        at[0].val.cooperative = 1;
        at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = at;
        cfg.numAttrs = 2;
        *fused_err = cudaLaunchKernelEx(&cfg, gdn_fused2_kernel<DK>, p);
        if (*fused_err != cudaSuccess) return;
    } else {
        configure_once<gdn_prep2_kernel<DK>>(PrepCfg<DK>::SMEM);
        launch_pdl(gdn_prep2_kernel<DK>, dim3(p.total_chunks * p.H), dim3(kPrepThreads), PrepCfg<DK>::SMEM, s, p);
        configure_once<gdn_chain2_kernel<DK>>(Chain2Cfg<DK>::SMEM);
        launch_pdl(gdn_chain2_kernel<DK>, dim3(p.dv / 32, p.H, p.n_chars), dim3(kThreads), Chain2Cfg<DK>::SMEM, s, p);
    }
    configure_once<gdn_out2_kernel<DK>>(Out2Cfg<DK>::SMEM);
    launch_pdl(gdn_out2_kernel<DK>, dim3(p.total_chunks * p.H), dim3(kThreads), Out2Cfg<DK>::SMEM, s, p);
}

}  // namespace

int64_t gdn_record_bytes(int dk, int dv) {
    const int64_t v1 = dk == 64 ? Rec<64>::bytes(dv) : Rec<128>::bytes(dv);
    return dk == 128 ? std::max<int64_t>(v1, Rec2<128>::bytes(dv)) : v1;   // a context may use either
}

int64_t gdn_snapshot_bytes(int dk, int dv) { return (int64_t)2 * dk * dv * 2; }

cudaError_t launch_gdn_v2(const GdnParams& p, int fused_grid, cudaStream_t s) {
    if (p.total_chunks <= 0) return cudaSuccess;
    if (p.dk != 128 || p.dv != 128 || p.dv_slice != 32) return cudaErrorInvalidValue;
    cudaError_t fe = cudaSuccess;
    launch_v2_dk<128>(p, fused_grid, s, &fe);
    return fe;
}

void launch_gdn_chunk_prep(const GdnParams& p, cudaStream_t s) {
    if (p.total_chunks <= 0) return;
    if (p.dk == 64) launch_prep_dk<64>(p, s);
    else if (p.dk == 128) launch_prep_dk<128>(p, s);
}

cudaError_t launch_gdn_fused(const GdnParams& p, int grid, cudaStream_t s) {
    if (p.total_chunks <= 0) return cudaSuccess;
    if (p.dv_slice > 32) return cudaErrorInvalidValue;    // the 512-thread blocks leave 128 registers a thread
    return p.dk == 64 ? launch_fused_dk<64>(p, grid, s) : launch_fused_dk<128>(p, grid, s);
}

void launch_gdn_chunk_scan(const GdnParams& p, cudaStream_t s) {
    if (p.total_chunks <= 0) return;
    if (p.dk == 64) launch_scan_dk<64>(p, s);
    else if (p.dk == 128) launch_scan_dk<128>(p, s);
}

}  // namespace kvm
