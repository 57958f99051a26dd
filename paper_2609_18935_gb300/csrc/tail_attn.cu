// True-tail prefill for one full-attention layer (Eq. 3, §4.2).
//
//  rope_append : rotate the tail's q and k at positions p + i (fp64 angle,
//                fp32 rotation), append rotated k and v at live slots L' + i
//                with their positions, and stage rotated q.
//  tail_attention : causal GQA attention of the tail's queries over the
//                compacted cache plus the tail itself.  A work item is
//                (character, KV head, 64-row query tile, key split); the 64
//                rows of a tile are (tail token, query head of the group)
//                pairs, token-major, so one K/V tile serves all g heads of
//                the group.  Online softmax in base 2; with one split the
//                normalised output is written directly, otherwise the
//                unnormalised partial accumulator and (max, sum) go to the
//                workspace and attn_combine merges the splits.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

constexpr int kRows = 64;      // query rows per tile
constexpr int kKeys = 64;      // keys per K/V tile
constexpr int kThreads = 256;

__global__ void __launch_bounds__(128) rope_append_kernel(const __grid_constant__ AttnParams p) {
    const int n = blockIdx.x;                 // packed tail token
    int lo = 0, hi = p.n_chars - 1;           // last b with tail_off <= n owns token n
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].tail_off <= n) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const AttnChar& c = p.ch[b];
    const int i = n - c.tail_off;
    if (i < 0 || i >= c.M) { if (threadIdx.x == 0) atomicOr(p.err, kErrBounds); return; }
    const int64_t pos = c.p + i;
    const int64_t slot = c.cap_off + c.L_prev + i;
    const int half = p.R / 2;

    __shared__ float cs[kMaxRotaryHalf], sn[kMaxRotaryHalf];
    for (int d = threadIdx.x; d < half; d += blockDim.x) {
        double sv, cv;
        sincos((double)pos * p.inv_freq[d], &sv, &cv);
        cs[d] = (float)cv;
        sn[d] = (float)sv;
    }
    __syncthreads();

    auto rotated = [&](const __nv_bfloat16* row, int d) -> float {
        const float x = __bfloat162float(row[d]);
        if (d >= p.R) return x;
        if (d < half) return x * cs[d] - __bfloat162float(row[d + half]) * sn[d];
        return x * cs[d - half] + __bfloat162float(row[d - half]) * sn[d - half];
    };

    for (int idx = threadIdx.x; idx < p.Hq * p.D; idx += blockDim.x) {
        const int h = idx / p.D, d = idx % p.D;
        const __nv_bfloat16* row = p.q + ((int64_t)n * p.Hq + h) * p.D;
        p.q_rot[((int64_t)n * p.Hq + h) * p.D + d] = __float2bfloat16_rn(rotated(row, d));
    }
    for (int idx = threadIdx.x; idx < p.Hkv * p.D; idx += blockDim.x) {
        const int h = idx / p.D, d = idx % p.D;
        const __nv_bfloat16* krow = p.k_new + ((int64_t)n * p.Hkv + h) * p.D;
        const int64_t dst = ((int64_t)h * p.slab_rows + slot) * p.D + d;
        p.K[dst] = __float2bfloat16_rn(rotated(krow, d));
        p.V[dst] = p.v_new[((int64_t)n * p.Hkv + h) * p.D + d];
    }
    if (threadIdx.x == 0) p.pos[slot] = (int32_t)pos;
}

// Work item -> (character, KV head, query tile, split).
__device__ __forceinline__ void decode_item(const AttnParams& p, int item, int& b, int& kvh,
                                            int& qt, int& sp) {
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
__global__ void __launch_bounds__(kThreads) tail_attention_kernel(const __grid_constant__ AttnParams p) {
    extern __shared__ float smem[];
    float* Qs = smem;                                   // [64][D]   rotated q * log2(e)/sqrt(D)
    float* Ss = Qs + kRows * D;                         // [64][65]  scores, then probabilities
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(Ss + kRows * (kKeys + 1));  // [64][D+2]
    __nv_bfloat16* Vs = Ks + kKeys * (D + 2);           // [64][D]
    __shared__ float row_m[kRows], row_l[kRows], row_a[kRows];
    __shared__ int row_lim[kRows];

    const int tid = threadIdx.x;
    const int item = blockIdx.x;
    int b, kvh, qt, sp;
    decode_item(p, item, b, kvh, qt, sp);
    const AttnChar& c = p.ch[b];
    const int g = p.g;
    const int tok0 = qt * p.tok_per_tile;
    const int tok_end = min(c.M, tok0 + p.tok_per_tile);
    const int n_keys = c.L_prev + tok_end;              // keys any row of this tile may see
    const int kt_total = (n_keys + kKeys - 1) / kKeys;
    const int kt0 = (int)((int64_t)sp * kt_total / p.n_split);
    const int kt1 = (int)((int64_t)(sp + 1) * kt_total / p.n_split);

    // load the query tile (rows past the tail reuse the last token; never stored)
    for (int idx = tid; idx < kRows * D; idx += kThreads) {
        const int r = idx / D, d = idx % D;
        const int tok = min(tok0 + r / g, c.M - 1);
        const int hq = kvh * g + (r % g);
        Qs[idx] = __bfloat162float(p.q_rot[((int64_t)(c.tail_off + tok) * p.Hq + hq) * D + d]) * p.scale_log2;
    }
    if (tid < kRows) {
        const int tok = min(tok0 + tid / g, c.M - 1);
        row_lim[tid] = c.L_prev + tok + 1;
        row_m[tid] = -INFINITY;
        row_l[tid] = 0.f;
    }

    const int ty = tid / 16, tx = tid % 16;
    constexpr int DJ = D / 16;
    float acc[4][DJ];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < DJ; ++j) acc[i][j] = 0.f;

    const __nv_bfloat16* Kbase = p.K + ((int64_t)kvh * p.slab_rows + c.cap_off) * D;
    const __nv_bfloat16* Vbase = p.V + ((int64_t)kvh * p.slab_rows + c.cap_off) * D;

    for (int kt = kt0; kt < kt1; ++kt) {
        __syncthreads();
        const int key0 = kt * kKeys;
        for (int idx = tid; idx < kKeys * (D / 8); idx += kThreads) {
            const int r = idx / (D / 8), d8 = (idx % (D / 8)) * 8;
            uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
            if (key0 + r < n_keys) {
                kv = *reinterpret_cast<const uint4*>(Kbase + (int64_t)(key0 + r) * D + d8);
                vv = *reinterpret_cast<const uint4*>(Vbase + (int64_t)(key0 + r) * D + d8);
            }
            const __nv_bfloat16* kh = reinterpret_cast<const __nv_bfloat16*>(&kv);
#pragma unroll
            for (int e = 0; e < 8; ++e) Ks[r * (D + 2) + d8 + e] = kh[e];
            *reinterpret_cast<uint4*>(Vs + r * D + d8) = vv;
        }
        __syncthreads();
        // scores for rows ty*4+i, keys tx + 16*j
        float s[4][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) s[i][j] = 0.f;
        for (int d = 0; d < D; ++d) {
            float qv[4], kv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) qv[i] = Qs[(ty * 4 + i) * D + d];
#pragma unroll
            for (int j = 0; j < 4; ++j) kv[j] = __bfloat162float(Ks[(tx + 16 * j) * (D + 2) + d]);
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) s[i][j] = fmaf(qv[i], kv[j], s[i][j]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int r = ty * 4 + i, key = tx + 16 * j;
                Ss[r * (kKeys + 1) + key] = (key0 + key < row_lim[r]) ? s[i][j] : -INFINITY;
            }
        __syncthreads();
        // online softmax: 4 threads per row
        {
            const int r = tid / 4, q4 = tid % 4;
            float mx = -INFINITY;
#pragma unroll
            for (int k = 0; k < 16; ++k) mx = fmaxf(mx, Ss[r * (kKeys + 1) + q4 + 4 * k]);
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
            const float m_old = row_m[r];
            const float m_new = fmaxf(m_old, mx);
            float sum = 0.f;
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                float* sp_ = &Ss[r * (kKeys + 1) + q4 + 4 * k];
                const float e = (m_new == -INFINITY) ? 0.f : exp2f(*sp_ - m_new);
                *sp_ = e;
                sum += e;
            }
            sum += __shfl_xor_sync(0xffffffffu, sum, 1);
            sum += __shfl_xor_sync(0xffffffffu, sum, 2);
            __syncwarp();
            if (q4 == 0) {
                const float a = (m_old == -INFINITY) ? 0.f : exp2f(m_old - m_new);
                row_a[r] = a;
                row_l[r] = row_l[r] * a + sum;
                row_m[r] = m_new;
            }
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float a = row_a[ty * 4 + i];
#pragma unroll
            for (int j = 0; j < DJ; ++j) acc[i][j] *= a;
        }
        for (int key = 0; key < kKeys; ++key) {
            float pv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) pv[i] = Ss[(ty * 4 + i) * (kKeys + 1) + key];
#pragma unroll
            for (int j = 0; j < DJ; ++j) {
                const float vv = __bfloat162float(Vs[key * D + tx + 16 * j]);
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[i][j] = fmaf(pv[i], vv, acc[i][j]);
            }
        }
    }
    __syncthreads();

#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = ty * 4 + i;
        const int tok = tok0 + r / g;
        if (tok >= c.M) continue;
        const int hq = kvh * g + (r % g);
        if (p.n_split == 1) {
            const float inv = 1.f / row_l[r];
            __nv_bfloat16* o = p.out + ((int64_t)(c.tail_off + tok) * p.Hq + hq) * D;
#pragma unroll
            for (int j = 0; j < DJ; ++j) o[tx + 16 * j] = __float2bfloat16_rn(acc[i][j] * inv);
        } else {
            float* o = p.part_o + ((int64_t)item * kRows + r) * D;
#pragma unroll
            for (int j = 0; j < DJ; ++j) o[tx + 16 * j] = acc[i][j];
            if (tx == 0) {
                p.part_ml[((int64_t)item * kRows + r) * 2 + 0] = row_m[r];
                p.part_ml[((int64_t)item * kRows + r) * 2 + 1] = row_l[r];
            }
        }
    }
}

// One block per (character, KV head, query tile): merge the key splits.
__global__ void __launch_bounds__(256) attn_combine_kernel(const __grid_constant__ AttnParams p) {
    const int tile = blockIdx.x;             // item index / n_split
    int b, kvh, qt, sp;
    decode_item(p, tile * p.n_split, b, kvh, qt, sp);
    const AttnChar& c = p.ch[b];
    const int item0 = tile * p.n_split;
    const int D = p.D;
    for (int idx = threadIdx.x; idx < kRows * D; idx += blockDim.x) {
        const int r = idx / D, d = idx % D;
        const int tok = qt * p.tok_per_tile + r / p.g;
        if (tok >= c.M) continue;
        float mx = -INFINITY;
        for (int s = 0; s < p.n_split; ++s)
            mx = fmaxf(mx, p.part_ml[((int64_t)(item0 + s) * kRows + r) * 2]);
        float num = 0.f, den = 0.f;
        for (int s = 0; s < p.n_split; ++s) {
            const float m = p.part_ml[((int64_t)(item0 + s) * kRows + r) * 2];
            if (m == -INFINITY) continue;
            const float w = exp2f(m - mx);
            num += w * p.part_o[((int64_t)(item0 + s) * kRows + r) * D + d];
            den += w * p.part_ml[((int64_t)(item0 + s) * kRows + r) * 2 + 1];
        }
        const int hq = kvh * p.g + (r % p.g);
        p.out[((int64_t)(c.tail_off + tok) * p.Hq + hq) * D + d] = __float2bfloat16_rn(num / den);
    }
}

template <int D>
void launch_attn_d(const AttnParams& p, cudaStream_t s) {
    const size_t smem = sizeof(float) * (kRows * D + kRows * (kKeys + 1)) +
                        sizeof(__nv_bfloat16) * (kKeys * (D + 2) + kKeys * D);
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(tail_attention_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        configured |= 1ull << (dev & 63);
    }
    tail_attention_kernel<D><<<p.n_items, kThreads, smem, s>>>(p);
}

}  // namespace

void launch_rope_append(const AttnParams& p, int total_tokens, cudaStream_t s) {
    if (total_tokens <= 0) return;
    rope_append_kernel<<<total_tokens, 128, 0, s>>>(p);
}

void launch_tail_attention(const AttnParams& p, cudaStream_t s) {
    if (p.n_items <= 0) return;
    switch (p.D) {
        case 64: launch_attn_d<64>(p, s); break;
        case 128: launch_attn_d<128>(p, s); break;
        case 256: launch_attn_d<256>(p, s); break;
        default: break;   // rejected on the host
    }
}

void launch_attn_combine(const AttnParams& p, int n_tiles, cudaStream_t s) {
    if (n_tiles <= 0 || p.n_split <= 1) return;
    attn_combine_kernel<<<n_tiles, 256, 0, s>>>(p);
}

}  // namespace kvm
