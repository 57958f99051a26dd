// Gated delta rule from the carried state on the sm_100-family tensor cores
// (Eq. 3 for a recurrent layer; Gated DeltaNet, the layer family of §4.1):
//     S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T,  o_t = S_t q_t.
//
// One block per (character, head, slice of d_v rows of S); 256 threads.  Warp
// w reads TMEM lanes 32*(w % 4) .. +31, so TMEM row r is shared by one thread
// of warp w and one of warp w + 4, which split its columns.  The state slice
// lives in TMEM as S^T (lanes = d_k index c, columns = d_v index r, fp32).
// Chunks of C = 64 tokens are processed in order.  With g_t = sum_{u<=t}
// log alpha_u, G_t = exp(g_t) and w_j = beta_j exp(g_C - g_j):
//   KK, QK   = [K;Q] K^T                                  (MMA)
//   L        = strict_lower(exp(g_t - g_j) beta_j KK),  A = lower(exp(g_t - g_j) beta_j QK)
//   X        = [I; A] (I + L)^-1 = [T; A T]                (per-row triangular solve, fp32)
//   W  = X G K,  U = X V  (rows 0..63: W, U; rows 64..127: A W, A U)       (MMA)
//   Q' = G Q - A W
//   [W S0^T; Q' S0^T] = [W; Q'] S0^T                      (MMA with the state)
//   E  = U - W S0^T,   O = A U + Q' S0^T  (= G Q S0^T + A E)
//   S^T = G_C S0^T + K^T diag(w) E                          (MMA, accumulated in TMEM)
// Tensor-core operands are bf16.  The inputs K, Q, V are exact in bf16 and
// are used in place (K and V as MN-major operands in their natural row
// layout).  Every computed fp32 operand x (X, W, Q', S, w E) is split into
// x_hi = bf16(x) and x_lo = bf16(x - x_hi); a product of two split operands
// is hi*hi + hi*lo + lo*hi with fp32 accumulation, about 2^-15 relative
// accuracy.  The master state stays fp32 in TMEM.
#include "kvm_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvm {
namespace {

using namespace ptx;

constexpr int C = 64;            // chunk length
constexpr int kThreads = 256;
constexpr int DVMAX = 128;       // d_v rows per block
constexpr int LSTRIDE = 68;      // fp32 row stride of the L scratch (conflict-free row vectors)

template <int DK>
struct GCfg {
    // byte offsets of the shared-memory regions (each 1024-aligned)
    static constexpr int KQ = 128 * DK * 2;                  // [K;Q] bf16, K-major, 128 rows
    static constexpr int V = C * DVMAX * 2;                  // V bf16, rows j (MN-major operand)
    static constexpr int TILE128 = 128 * 64 * 2;             // 128 x 64 bf16 K-major tile (16 KB)
    static constexpr int WQ = 2 * 128 * DK * 2;              // [W;Q'] hi, lo
    static constexpr int RA = (WQ > 32768 + 2 * TILE128) ? WQ : 32768 + 2 * TILE128;   // L + X*G hi/lo, then [W;Q']
    static constexpr int RX = 2 * TILE128;                   // X hi, lo
    static constexpr int RS = 2 * DK * DVMAX * 2;            // S hi, lo (rows c); w E hi, lo aliased
    static constexpr int OFF_KQ = 0;
    static constexpr int OFF_V = OFF_KQ + KQ;
    static constexpr int OFF_A = OFF_V + V;
    static constexpr int OFF_X = OFF_A + RA;
    static constexpr int OFF_S = OFF_X + RX;
    static constexpr int OFF_BAR = OFF_S + RS;
    static constexpr int SMEM = OFF_BAR + 64 + 1024;
    // TMEM columns
    static constexpr uint32_t T_D = 0;          // KK/QK (64 cols), later [W;Q'] S0^T (dv cols)
    static constexpr uint32_t T_WU = 128;       // [W | U] (DK + dv cols)
    static constexpr uint32_t T_S = 384;        // S^T     (dv cols)
};

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

template <int DK>
__global__ void __launch_bounds__(kThreads, 1) gdn_chunk_tc_kernel(const __grid_constant__ GdnParams p) {
    using G = GCfg<DK>;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment by pointer arithmetic on the shared array, so that the
    // accesses below stay shared-memory accesses
    uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sb = smem_u32(smem);
    auto V4 = [&](uint32_t off) -> uint4& { return *reinterpret_cast<uint4*>(smem + off); };
    constexpr uint32_t oKQ = G::OFF_KQ, oV = G::OFF_V, oA = G::OFF_A, oX = G::OFF_X, oS = G::OFF_S;
    constexpr uint32_t oL = oA;                                  // fp32 [64][LSTRIDE]
    constexpr uint32_t oXG = oA + 32768;                         // X G hi, lo (K-major 128 x 64)
    constexpr uint32_t T128 = G::TILE128;
    constexpr uint32_t WQH = 128 * DK * 2;                       // one [W;Q'] half
    constexpr uint32_t SH = DK * DVMAX * 2;                      // one S half
    constexpr uint32_t WEH = C * DVMAX * 2;                      // one w E half
    float* Lm = reinterpret_cast<float*>(smem + oL);
    uint64_t* bar = reinterpret_cast<uint64_t*>(smem + G::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + G::OFF_BAR + 8);
    const uint32_t mbar = smem_u32(bar);
    __shared__ float gs[C], bs[C], Gs[C], ws[C];
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int q4 = warp & 3, hf = warp >> 2;
    const int row = q4 * 32 + lane;                  // TMEM lane owned (with its twin in warp w ^ 4)
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const int dvs = p.dv_slice;
    const int r0 = blockIdx.x * dvs;
    const int h = blockIdx.y;
    const int b = blockIdx.z;
    const GdnChar ch = p.ch[b];
    if (ch.M <= 0) return;                           // uniform per block
    const int H = p.H, dv = p.dv;
    float* Sg = p.S + ((int64_t)b * H + h) * dv * DK;
    // columns of a dv-wide TMEM row handled by this thread: [dlo, dhi)
    const int dhalf = ((dvs / 2) + 31) / 32 * 32;
    const int dlo = hf * dhalf, dhi = min(dvs, dlo + dhalf);

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(mbar, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    // S operand (MN-major: row c, column r) from fp32 values of row c
    auto write_s_row = [&](int c, int rc, const float* x) {
#pragma unroll
        for (int j8 = 0; j8 < 32; j8 += 8) {
            if (rc + j8 < dvs) {
                uint4 hi, lo;
                split8(x + j8, hi, lo);
                const uint32_t off = sw128_off16(c, rc + j8, DK);
                V4(oS + off) = hi;
                V4(oS + SH + off) = lo;
            }
        }
    };

    // ---- load the state slice: S^T into TMEM (lane c, column r) and the operand
    for (int rc = dlo; rc < dhi; rc += 32) {
        uint32_t v[32];
        float x[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int r = rc + j;
            x[j] = (row < DK && r < dvs) ? Sg[(int64_t)(r0 + r) * DK + row] : 0.f;
            v[j] = __float_as_uint(x[j]);
        }
        tmem_st32(tmem + lane_off + G::T_S + rc, v);
        if (row < DK) write_s_row(row, rc, x);
    }
    tmem_st_wait();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();

    uint32_t phase = 0;
    bool ok = true;
    auto mma_wait = [&]() -> bool {
        bool r = mbar_wait(mbar, phase, &abort_flag, p.err, kErrWait);
        phase ^= 1;
        r = __syncthreads_and(r);
        tc_fence_after();
        return r;
    };
    auto issue_begin = [&]() { fence_proxy_async_smem(); tc_fence_before(); __syncthreads(); };
    const uint32_t id_kk = idesc_bf16_f32(128, C, false);
    const uint32_t id_w = idesc_bf16_f32(128, DK, true);            // B = K, MN-major
    const uint32_t id_u = idesc_bf16_f32(128, dvs, true);           // B = V, MN-major
    const uint32_t id_1 = idesc_bf16_f32(128, dvs, true);           // B = S, MN-major
    const uint32_t id_2 = idesc_bf16_f32(128, dvs, true, true);     // A = K, B = w E, both MN-major
    const uint32_t kq_region = 128 * 128;                           // [K;Q] region stride (64 columns)

    for (int c0 = 0; c0 < ch.M && ok; c0 += C) {
        const int n = min(C, ch.M - c0);
        const int64_t tok0 = ch.tail_off + c0;
        // ---------------------------------------------------------------- loads
        for (int i = tid; i < 128 * (DK / 8); i += kThreads) {
            const int rr = i / (DK / 8), c8 = (i % (DK / 8)) * 8;
            const int t = rr & 63;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (t < n) v = *reinterpret_cast<const uint4*>((rr < 64 ? p.k : p.q) + ((tok0 + t) * H + h) * DK + c8);
            V4(oKQ + sw128_off16(rr, c8, 128)) = v;
        }
        for (int i = tid; i < C * (dvs / 8); i += kThreads) {
            const int t = i / (dvs / 8), r8 = (i % (dvs / 8)) * 8;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (t < n) v = *reinterpret_cast<const uint4*>(p.v + ((tok0 + t) * H + h) * dv + r0 + r8);
            V4(oV + sw128_off16(t, r8, C)) = v;
        }
        if (tid < 32) {
            float x0 = tid < n ? logf(p.alpha[(tok0 + tid) * H + h]) : 0.f;
            float x1 = tid + 32 < n ? logf(p.alpha[(tok0 + tid + 32) * H + h]) : 0.f;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y0 = __shfl_up_sync(0xffffffffu, x0, o);
                const float y1 = __shfl_up_sync(0xffffffffu, x1, o);
                if (tid >= o) { x0 += y0; x1 += y1; }
            }
            x1 += __shfl_sync(0xffffffffu, x0, 31);
            gs[tid] = x0;
            gs[tid + 32] = x1;
            bs[tid] = tid < n ? p.beta[(tok0 + tid) * H + h] : 0.f;
            bs[tid + 32] = tid + 32 < n ? p.beta[(tok0 + tid + 32) * H + h] : 0.f;
        }
        issue_begin();
        if (tid < C) {
            Gs[tid] = expf(gs[tid]);
            ws[tid] = tid < n ? bs[tid] * expf(gs[n - 1] - gs[tid]) : 0.f;
        }
        // ---------------------------------------------------------------- KK, QK
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t off = (ks >> 2) * kq_region + (ks & 3) * 32;
                mma_bf16(tmem + G::T_D, smem_desc_sw128(sb + oKQ + off, 16, 1024),
                         smem_desc_sw128(sb + oKQ + off, 16, 1024), id_kk, ks > 0);
            }
            mma_commit(mbar);
        }
        ok = mma_wait();                            // also publishes Gs, ws
        if (!ok) break;
        // ---------------------------------------------------------------- L, A; X = [I; A] (I + L)^-1
        float x[C];
        if (hf == 0) {
            uint32_t v0[32], v1[32];
            tmem_ld32(tmem + lane_off + G::T_D, v0);
            tmem_ld32(tmem + lane_off + G::T_D + 32, v1);
            tmem_ld_wait();
            const int t = row & 63;
            const float gt = gs[t];
#pragma unroll
            for (int j = 0; j < C; ++j) {
                const float d = __uint_as_float(j < 32 ? v0[j] : v1[j - 32]);
                const bool keep = (row < 64) ? (j < t) : (j <= t);
                x[j] = (keep && t < n) ? expf(gt - gs[j]) * bs[j] * d : 0.f;
            }
            if (row < 64) {
#pragma unroll
                for (int j = 0; j < C; j += 4)
                    *reinterpret_cast<float4*>(Lm + t * LSTRIDE + j) = make_float4(x[j], x[j + 1], x[j + 2], x[j + 3]);
#pragma unroll
                for (int j = 0; j < C; ++j) x[j] = (j == t) ? 1.f : 0.f;       // right-hand side e_t
            }
        }
        __syncthreads();
        if (hf == 0) {
            // x (I + L) = b, L strictly lower: x_j = b_j - sum_{i>j} x_i L[i][j]
#pragma unroll
            for (int i = C - 1; i > 0; --i) {
                const float xi = x[i];
#pragma unroll
                for (int j4 = 0; j4 < i; j4 += 4) {
                    const float4 l4 = *reinterpret_cast<const float4*>(Lm + i * LSTRIDE + j4);
                    x[j4] = fmaf(-xi, l4.x, x[j4]);
                    if (j4 + 1 < i) x[j4 + 1] = fmaf(-xi, l4.y, x[j4 + 1]);
                    if (j4 + 2 < i) x[j4 + 2] = fmaf(-xi, l4.z, x[j4 + 2]);
                    if (j4 + 3 < i) x[j4 + 3] = fmaf(-xi, l4.w, x[j4 + 3]);
                }
            }
        }
        __syncthreads();                             // every row finished reading L
        if (hf == 0) {
            // operands: X G (for W) and X (for U), K-major rows
#pragma unroll
            for (int j8 = 0; j8 < C; j8 += 8) {
                float xg[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) xg[e] = x[j8 + e] * Gs[j8 + e];
                uint4 hi, lo;
                split8(xg, hi, lo);
                const uint32_t off = sw128_off16(row, j8, 128);
                V4(oXG + off) = hi;
                V4(oXG + T128 + off) = lo;
                split8(x + j8, hi, lo);
                V4(oX + off) = hi;
                V4(oX + T128 + off) = lo;
            }
        }
        issue_begin();
        // ---------------------------------------------------------------- [W | U] = X [G K | V]
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < C / 16; ++ks) {
                const uint64_t bk = smem_desc_sw128(sb + oKQ + ks * 2048, kq_region, 1024);
                const uint64_t bvv = smem_desc_sw128(sb + oV + ks * 2048, C * 128, 1024);
#pragma unroll
                for (int part = 0; part < 2; ++part) {
                    const uint32_t ao = part * T128 + ks * 32;
                    mma_bf16(tmem + G::T_WU, smem_desc_sw128(sb + oXG + ao, 16, 1024), bk, id_w, (ks | part) != 0);
                    mma_bf16(tmem + G::T_WU + DK, smem_desc_sw128(sb + oX + ao, 16, 1024), bvv, id_u,
                             (ks | part) != 0);
                }
            }
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        // ---------------------------------------------------------------- [W; Q'] operand (hi, lo)
        {
            const int t = row & 63;
            const float gt = Gs[t];
            for (int cb = hf * (DK / 2); cb < (hf + 1) * (DK / 2); cb += 32) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_off + G::T_WU + cb, v);
                tmem_ld_wait();
                float y[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) y[j] = __uint_as_float(v[j]);
                if (row >= 64) {
                    // Q' = G Q - A W ; row `row` of [K;Q] holds q_t
#pragma unroll
                    for (int j8 = 0; j8 < 32; j8 += 8) {
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
                for (int j8 = 0; j8 < 32; j8 += 8) {
                    uint4 hi, lo;
                    split8(y + j8, hi, lo);
                    const uint32_t off = sw128_off16(row, cb + j8, 128);
                    V4(oA + off) = hi;
                    V4(oA + WQH + off) = lo;
                }
            }
        }
        issue_begin();
        // ---------------------------------------------------------------- [W; Q'] S0^T
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < DK / 16; ++ks) {
                const uint32_t ao = (ks >> 2) * kq_region + (ks & 3) * 32;
                const uint32_t bo = ks * 2048;
                const uint64_t a_hi = smem_desc_sw128(sb + oA + ao, 16, 1024);
                const uint64_t a_lo = smem_desc_sw128(sb + oA + WQH + ao, 16, 1024);
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
        // ---------------------------------------------------------------- E, O; S^T *= G_C
        {
            const int t = row & 63;
            const float gC = expf(gs[n - 1]);
            const float wt = ws[t];
            for (int rc = dlo; rc < dhi; rc += 32) {
                uint32_t d1[32], u[32], sv[32];
                tmem_ld32(tmem + lane_off + G::T_D + rc, d1);
                tmem_ld32(tmem + lane_off + G::T_WU + DK + rc, u);
                tmem_ld32(tmem + lane_off + G::T_S + rc, sv);
                tmem_ld_wait();
                if (row < 64) {
                    float e[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) e[j] = wt * (__uint_as_float(u[j]) - __uint_as_float(d1[j]));
#pragma unroll
                    for (int j8 = 0; j8 < 32; j8 += 8) {
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
                    for (int j8 = 0; j8 < 32; j8 += 8) {
                        if (rc + j8 < dvs) {
                            uint4 w4;
                            uint32_t* ww = reinterpret_cast<uint32_t*>(&w4);
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                ww[e] = pack_bf16x2(__uint_as_float(u[j8 + 2 * e]) + __uint_as_float(d1[j8 + 2 * e]),
                                                    __uint_as_float(u[j8 + 2 * e + 1]) + __uint_as_float(d1[j8 + 2 * e + 1]));
                            *reinterpret_cast<uint4*>(o + j8) = w4;
                        }
                    }
                }
#pragma unroll
                for (int j = 0; j < 32; ++j) sv[j] = __float_as_uint(__uint_as_float(sv[j]) * gC);
                tmem_st32(tmem + lane_off + G::T_S + rc, sv);
            }
            tmem_st_wait();
        }
        issue_begin();
        // ---------------------------------------------------------------- S^T += K^T (w E)
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < C / 16; ++ks) {
                const uint64_t a = smem_desc_sw128(sb + oKQ + ks * 2048, kq_region, 1024);
                mma_bf16(tmem + G::T_S, a, smem_desc_sw128(sb + oS + ks * 2048, C * 128, 1024), id_2, 1u);
                mma_bf16(tmem + G::T_S, a, smem_desc_sw128(sb + oS + WEH + ks * 2048, C * 128, 1024), id_2, 1u);
            }
            mma_commit(mbar);
        }
        ok = mma_wait();
        if (!ok) break;
        // ---------------------------------------------------------------- refresh the state operand
        for (int rc = dlo; rc < dhi; rc += 32) {
            uint32_t sv[32];
            tmem_ld32(tmem + lane_off + G::T_S + rc, sv);
            tmem_ld_wait();
            if (row < DK) {
                float y[32];
#pragma unroll
                for (int j = 0; j < 32; ++j) y[j] = __uint_as_float(sv[j]);
                write_s_row(row, rc, y);
            }
        }
        issue_begin();
    }
    // ---- write the state slice back
    if (ok) {
        for (int rc = dlo; rc < dhi; rc += 32) {
            uint32_t sv[32];
            tmem_ld32(tmem + lane_off + G::T_S + rc, sv);
            tmem_ld_wait();
            if (row < DK) {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (rc + j < dvs) Sg[(int64_t)(r0 + rc + j) * DK + row] = __uint_as_float(sv[j]);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

template <int DK>
void launch_gdn_tc_dk(const GdnParams& p, cudaStream_t s) {
    using G = GCfg<DK>;
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(gdn_chunk_tc_kernel<DK>, cudaFuncAttributeMaxDynamicSharedMemorySize, G::SMEM);
        configured |= 1ull << (dev & 63);
    }
    dim3 grid(p.dv / p.dv_slice, p.H, p.n_chars);
    gdn_chunk_tc_kernel<DK><<<grid, kThreads, G::SMEM, s>>>(p);
}

}  // namespace

void launch_gdn_chunk_scan(const GdnParams& p, cudaStream_t s) {
    if (p.dk == 64) launch_gdn_tc_dk<64>(p, s);
    else if (p.dk == 128) launch_gdn_tc_dk<128>(p, s);
}

}  // namespace kvm
