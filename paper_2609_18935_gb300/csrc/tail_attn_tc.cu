// Causal GQA attention of the true tail over the compacted cache (Eq. 3 for a
// full-attention layer), on the sm_100-family tensor cores.
//
// Work item = (character, KV head, 128-row query tile, key split).  The 128
// rows are (tail token, query head of the GQA group) pairs, token-major, so
// every K/V tile serves all g heads of the group.  Per item:
//   warp 0      TMA producer: Q tile once, then K and V tiles of 64 keys into
//               a two-stage ring (128-byte swizzled, K-major rows of head_dim);
//   warp 1      allocates TMEM; lane 0 issues tcgen05.mma:
//                 S_i = Q K_i^T   (M 128, N 64, K D)   -> TMEM, double-buffered
//                 O  += P_i V_i   (M 128, N D, K 64)   -> TMEM accumulator
//               S_{i+1} is issued before PV_i so it overlaps the softmax of i;
//   warps 2-5   one query row per thread: read S_i from TMEM, mask, online
//               softmax in base 2 with lazy rescaling (the running reference
//               max moves only when a score exceeds it by more than 2^8, and
//               then the O row in TMEM is rescaled), write P_i as bf16 into
//               shared memory in the MMA's swizzled K-major layout; finally
//               read O, normalise and store (or store the partial for the
//               split-combine).
// Every mbarrier wait is bounded; on expiry the block raises an abort flag,
// records kErrWait, drains its own copies and MMAs, frees TMEM and returns.
#include "kvm_internal.cuh"
#include "sm100_ptx.cuh"

namespace kvm {
namespace {

using namespace ptx;

constexpr int BM = 128;          // query rows per tile
constexpr int BN = 64;           // keys per K/V tile
constexpr int kThreads = 192;    // 6 warps

enum Bar { Q_FULL = 0, K_FULL = 1, K_EMPTY = 3, V_FULL = 5, V_EMPTY = 7, S_FULL = 9, S_EMPTY = 11,
           P_FULL = 13, PV_DONE = 14, O_FINAL = 15, N_BARS = 16 };

template <int D>
struct Cfg {
    static constexpr int NREG = D / 64;                    // 64-column (128-byte) regions
    static constexpr int Q_BYTES = BM * D * 2;
    static constexpr int KV_BYTES = BN * D * 2;
    static constexpr int P_BYTES = BM * BN * 2;
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_K = OFF_Q + Q_BYTES;
    static constexpr int OFF_V = OFF_K + 2 * KV_BYTES;
    static constexpr int OFF_P = OFF_V + 2 * KV_BYTES;
    static constexpr int OFF_BAR = OFF_P + P_BYTES;
    static constexpr int USED = OFF_BAR + N_BARS * 8 + 16;
    // D = 64 would fit three blocks per SM by shared memory but TMEM holds two
    static constexpr int SMEM = (USED + 1024 > 80 * 1024 || D != 64) ? USED + 1024 : 80 * 1024;
    static constexpr uint32_t TMEM_S = 0;                  // two S buffers of BN columns
    static constexpr uint32_t TMEM_O = 2 * BN;             // D columns
    static constexpr uint32_t TMEM_COLS = (2 * BN + D <= 256) ? 256 : 512;
};

__device__ __forceinline__ void decode_item(const AttnParams& p, int item, int& b, int& kvh, int& qt, int& sp) {
    int lo = 0, hi = p.n_chars - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].item_off <= item) lo = mid; else hi = mid - 1;
    }
    b = lo;
    int local = item - p.ch[b].item_off;
    sp = local % p.n_split;
    local /= p.n_split;
    qt = local % p.ch[b].n_qtiles;
    kvh = local / p.ch[b].n_qtiles;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1) tail_attention_tc_kernel(const __grid_constant__ AttnParams p) {
    using C = Cfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(smem);
    const uint32_t sQ = sbase + C::OFF_Q, sK = sbase + C::OFF_K, sV = sbase + C::OFF_V, sP = sbase + C::OFF_P;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_BAR + N_BARS * 8);
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int b, kvh, qt, sp;
    decode_item(p, blockIdx.x, b, kvh, qt, sp);
    const AttnChar& c = p.ch[b];
    const int g = p.g;
    const int tok0 = qt * p.tok_per_tile;
    const int tok_end = min(c.M, tok0 + p.tok_per_tile);
    const int n_keys = c.L_prev + tok_end;
    const int kt_total = (n_keys + BN - 1) / BN;
    const int kt0 = (int)((int64_t)sp * kt_total / p.n_split);
    const int kt1 = (int)((int64_t)(sp + 1) * kt_total / p.n_split);
    const int n = kt1 - kt0;
    const int key_row0 = (p.attn_layer * p.Hkv + kvh) * (int)p.slab_rows + c.cap_off;

    if (tid == 0) {
        abort_flag = 0;
        mbar_init(bar(Q_FULL), 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(bar(K_FULL + s), 1);
            mbar_init(bar(K_EMPTY + s), 1);
            mbar_init(bar(V_FULL + s), 1);
            mbar_init(bar(V_EMPTY + s), 1);
            mbar_init(bar(S_FULL + s), 1);
            mbar_init(bar(S_EMPTY + s), 128);
        }
        mbar_init(bar(P_FULL), 128);
        mbar_init(bar(PV_DONE), 1);
        mbar_init(bar(O_FINAL), 1);
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

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0 && n > 0) {
            prefetch_tmap(&p.tmap_q);
            prefetch_tmap(&p.tmap_k);
            prefetch_tmap(&p.tmap_v);
            mbar_arrive_expect_tx(bar(Q_FULL), C::Q_BYTES);
            for (int r = 0; r < C::NREG; ++r)
                tma_load_3d(sQ + r * (BM * 128), &p.tmap_q, r * 64, kvh * g, c.tail_off + tok0, bar(Q_FULL));
            int issued_k[2] = {-1, -1}, issued_v[2] = {-1, -1};
            bool ok = true;
            for (int i = 0; i < n && ok; ++i) {
                const int st = i & 1;
                const int row = key_row0 + (kt0 + i) * BN;
                if (i >= 2) ok = mbar_wait(bar(K_EMPTY + st), ((i >> 1) - 1) & 1, &abort_flag, p.err, kErrWait, p.diag, 0x10 + K_EMPTY + 256 * i);
                if (!ok) break;
                mbar_arrive_expect_tx(bar(K_FULL + st), C::KV_BYTES);
                for (int r = 0; r < C::NREG; ++r)
                    tma_load_2d(sK + st * C::KV_BYTES + r * (BN * 128), &p.tmap_k, r * 64, row, bar(K_FULL + st));
                issued_k[st] = i;
                if (i >= 2) ok = mbar_wait(bar(V_EMPTY + st), ((i >> 1) - 1) & 1, &abort_flag, p.err, kErrWait, p.diag, 0x10 + V_EMPTY + 256 * i);
                if (!ok) break;
                mbar_arrive_expect_tx(bar(V_FULL + st), C::KV_BYTES);
                for (int r = 0; r < C::NREG; ++r)
                    tma_load_2d(sV + st * C::KV_BYTES + r * (BN * 128), &p.tmap_v, r * 64, row, bar(V_FULL + st));
                issued_v[st] = i;
            }
            if (abort_flag) {
                // drain this block's own copies before the block exits
                volatile int never = 0;
                mbar_wait(bar(Q_FULL), 0, &never, p.err, kErrWait);
                for (int s = 0; s < 2; ++s) {
                    if (issued_k[s] >= 0) mbar_wait(bar(K_FULL + s), (issued_k[s] >> 1) & 1, &never, p.err, kErrWait);
                    if (issued_v[s] >= 0) mbar_wait(bar(V_FULL + s), (issued_v[s] >> 1) & 1, &never, p.err, kErrWait);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && n > 0) {
            const uint32_t id_qk = idesc_bf16_f32(BM, BN, false);
            const uint32_t id_pv = idesc_bf16_f32(BM, D, true);
            auto issue_s = [&](int i) -> bool {
                const int st = i & 1;
                if (!mbar_wait(bar(K_FULL + st), (i >> 1) & 1, &abort_flag, p.err, kErrWait, p.diag, 0x20 + K_FULL + 256 * i)) return false;
                if (i >= 2 && !mbar_wait(bar(S_EMPTY + st), ((i >> 1) - 1) & 1, &abort_flag, p.err, kErrWait, p.diag, 0x20 + S_EMPTY + 256 * i))
                    return false;
                tc_fence_after();
                const uint32_t kb = sK + st * C::KV_BYTES;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const uint64_t ad = smem_desc_sw128(sQ + (ks >> 2) * (BM * 128) + (ks & 3) * 32, 16, 1024);
                    const uint64_t bd = smem_desc_sw128(kb + (ks >> 2) * (BN * 128) + (ks & 3) * 32, 16, 1024);
                    mma_bf16(tmem + C::TMEM_S + st * BN, ad, bd, id_qk, ks > 0);
                }
                mma_commit(bar(S_FULL + st));
                mma_commit(bar(K_EMPTY + st));
                return true;
            };
            auto issue_pv = [&](int i) -> bool {
                const int st = i & 1;
                if (!mbar_wait(bar(P_FULL), i & 1, &abort_flag, p.err, kErrWait, p.diag, 0x20 + P_FULL + 256 * i)) return false;
                if (!mbar_wait(bar(V_FULL + st), (i >> 1) & 1, &abort_flag, p.err, kErrWait, p.diag, 0x20 + V_FULL + 256 * i)) return false;
                tc_fence_after();
                const uint32_t vb = sV + st * C::KV_BYTES;
#pragma unroll
                for (int ks = 0; ks < BN / 16; ++ks) {
                    const uint64_t ad = smem_desc_sw128(sP + ks * 32, 16, 1024);
                    const uint64_t bd = smem_desc_sw128(vb + ks * 16 * 128, BN * 128, 1024);
                    mma_bf16(tmem + C::TMEM_O, ad, bd, id_pv, (i > 0 || ks > 0) ? 1u : 0u);
                }
                mma_commit(bar(PV_DONE));
                mma_commit(bar(V_EMPTY + st));
                return true;
            };
            bool ok = mbar_wait(bar(Q_FULL), 0, &abort_flag, p.err, kErrWait, p.diag, 0x20 + Q_FULL);
            if (ok) ok = issue_s(0);
            for (int i = 0; i < n && ok; ++i) {
                if (i + 1 < n) ok = issue_s(i + 1);
                if (ok) ok = issue_pv(i);
            }
            // every MMA issued by this thread completes before O_FINAL arrives
            mma_commit(bar(O_FINAL));
            volatile int never = 0;
            mbar_wait(bar(O_FINAL), 0, &never, p.err, kErrWait);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        const int quarter = warp & 3;                    // TMEM lanes 32*quarter .. +31
        const int r = quarter * 32 + lane;               // query row of this thread
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        const int tok = tok0 + r / g;
        const bool row_valid = tok < c.M;
        const int lim = c.L_prev + min(tok, c.M - 1) + 1;     // keys [0, lim) are visible
        const float sl = p.scale_log2;
        float mr = -INFINITY;                            // reference max, log2 units
        float l = 0.f;
        bool ok = true;
        // waits are made warp-uniform so that an abort never splits a warp
        // before the warp-collective tcgen05.ld / tcgen05.st below
        auto wait_all = [&](int which, uint32_t parity) -> bool {
            const bool r = mbar_wait(bar(which), parity, &abort_flag, p.err, kErrWait, p.diag, 0x30 + which);
            return __all_sync(0xffffffffu, r);
        };
        for (int i = 0; i < n && ok; ++i) {
            const int st = i & 1;
            ok = wait_all(S_FULL + st, (i >> 1) & 1);
            if (!ok) break;
            tc_fence_after();
            uint32_t sa[32], sb[32];
            tmem_ld32(tmem + lane_off + C::TMEM_S + st * BN, sa);
            tmem_ld32(tmem + lane_off + C::TMEM_S + st * BN + 32, sb);
            tmem_ld_wait();
            tc_fence_before();
            mbar_arrive(bar(S_EMPTY + st));
            float s[64];
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                s[j] = __uint_as_float(sa[j]);
                s[32 + j] = __uint_as_float(sb[j]);
            }
            const int key0 = (kt0 + i) * BN;
            if (key0 + BN > lim) {
#pragma unroll
                for (int j = 0; j < 64; ++j)
                    if (key0 + j >= lim) s[j] = -INFINITY;
            }
            float mx = s[0];
#pragma unroll
            for (int j = 1; j < 64; ++j) mx = fmaxf(mx, s[j]);
            const float mx2 = mx * sl;
            const bool bump = mx2 > mr + 8.0f;           // also true while mr = -inf and a key is visible
            const float mr_new = bump ? mx2 : mr;
            float pv[64];
            float sum = 0.f;
            if (mr_new == -INFINITY) {
#pragma unroll
                for (int j = 0; j < 64; ++j) pv[j] = 0.f;
            } else {
#pragma unroll
                for (int j = 0; j < 64; ++j) {
                    pv[j] = ex2(fmaf(s[j], sl, -mr_new));
                    sum += pv[j];
                }
            }
            const float factor = bump ? ((mr == -INFINITY) ? 0.f : ex2(mr - mr_new)) : 1.f;
            // P buffer and O are free once the previous PV has completed
            if (i > 0) {
                ok = wait_all(PV_DONE, (i - 1) & 1);
                if (!ok) break;
                tc_fence_after();
                if (__any_sync(0xffffffffu, bump)) {
#pragma unroll 1
                    for (int c0 = 0; c0 < D; c0 += 32) {
                        uint32_t o[32];
                        tmem_ld32(tmem + lane_off + C::TMEM_O + c0, o);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * factor);
                        tmem_st32(tmem + lane_off + C::TMEM_O + c0, o);
                    }
                    tmem_st_wait();
                }
            }
            l = l * factor + sum;
            mr = mr_new;
            // P row r: 64 bf16 = 8 chunks of 16 bytes, chunk index XOR (row & 7)
#pragma unroll
            for (int ch = 0; ch < 8; ++ch) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    __nv_bfloat162 h2 = __floats2bfloat162_rn(pv[ch * 8 + 2 * e], pv[ch * 8 + 2 * e + 1]);
                    w[e] = *reinterpret_cast<uint32_t*>(&h2);
                }
                st_shared_v4(sP + r * 128 + ((ch ^ (r & 7)) << 4), w[0], w[1], w[2], w[3]);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(bar(P_FULL));
        }
        if (n > 0 && ok) ok = wait_all(O_FINAL, 0);
        if (ok) {
            tc_fence_after();
            const int hq = kvh * g + (r % g);
            const int64_t item_row = (int64_t)blockIdx.x * BM + r;
            if (p.n_split == 1) {
                // tcgen05.ld is warp-collective (.sync.aligned): every lane
                // loads, and only lanes of real query rows store
                const float inv = row_valid ? 1.f / l : 0.f;
                __nv_bfloat16* o = p.out + ((int64_t)(c.tail_off + (row_valid ? tok : 0)) * p.Hq + hq) * D;
#pragma unroll 1
                for (int c0 = 0; c0 < D; c0 += 32) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + C::TMEM_O + c0, v);
                    tmem_ld_wait();
                    if (row_valid) {
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
                p.part_ml[item_row * 2 + 0] = mr;
                p.part_ml[item_row * 2 + 1] = l;
                if (n > 0) {
                    float* o = p.part_o + item_row * D;
#pragma unroll 1
                    for (int c0 = 0; c0 < D; c0 += 32) {
                        uint32_t v[32];
                        tmem_ld32(tmem + lane_off + C::TMEM_O + c0, v);
                        tmem_ld_wait();
                        uint4* dst = reinterpret_cast<uint4*>(o + c0);
#pragma unroll
                        for (int e = 0; e < 8; ++e) dst[e] = make_uint4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
                    }
                }
            }
        }
        tc_fence_before();
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
    tail_attention_tc_kernel<D><<<p.n_items, kThreads, C::SMEM, s>>>(p);
}

}  // namespace

void launch_tail_attention(const AttnParams& p, cudaStream_t s) {
    if (p.n_items <= 0) return;
    switch (p.D) {
        case 64: launch_tc<64>(p, s); break;
        case 128: launch_tc<128>(p, s); break;
        case 256: launch_tc<256>(p, s); break;
        default: break;   // rejected on the host
    }
}

int attention_rows_per_tile() { return BM; }

}  // namespace kvm
