// True-tail prefill for one full-attention layer (Eq. 3, §4.2): the kernels
// around the tensor-core attention (tail_attn_tc.cu).
//
//  rope_append : rotate the tail's q and k at positions p + i, append the
//                rotated k and v at live slots L' + i with their positions,
//                and stage the rotated q for the attention's TMA loads.
//                The angle pos * omega_d is formed and reduced modulo 2*pi in
//                fp64 (positions far beyond the live length stay accurate),
//                then sin/cos and the rotation run in fp32.
//  attn_combine : merge the key splits of the attention: each split leaves
//                an unnormalised accumulator and (reference max in log2
//                units, sum); one warp per query row.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

constexpr int kRows = kAttnRows;   // query rows per attention work item
constexpr double kTwoPi = 6.283185307179586476925286766559;

__device__ __forceinline__ float2 bf2_to_f2(uint32_t w) {
    __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&w);
    return __bfloat1622float2(h);
}
__device__ __forceinline__ uint32_t f2_to_bf2(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

// Rotate 8 pairs (lo[e], hi[e]) by the angles of dims d0 .. d0+7.
__device__ __forceinline__ void rotate8(uint4& lo, uint4& hi, const float* cs, const float* sn, int d0) {
    uint32_t* L = reinterpret_cast<uint32_t*>(&lo);
    uint32_t* Hh = reinterpret_cast<uint32_t*>(&hi);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float2 x = bf2_to_f2(L[e]), y = bf2_to_f2(Hh[e]);
        const int d = d0 + 2 * e;
        const float c0 = cs[d], s0 = sn[d], c1 = cs[d + 1], s1 = sn[d + 1];
        L[e] = f2_to_bf2(x.x * c0 - y.x * s0, x.y * c1 - y.y * s1);
        Hh[e] = f2_to_bf2(y.x * c0 + x.x * s0, y.y * c1 + x.y * s1);
    }
}

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
    const int D = p.D;

    __shared__ float cs[kMaxRotaryHalf], sn[kMaxRotaryHalf];
    for (int d = threadIdx.x; d < half; d += blockDim.x) {
        const double ang = (double)pos * p.inv_freq[d];
        const double r = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);   // ang mod 2*pi, |r| <= pi
        float sv, cv;
        sincosf((float)r, &sv, &cv);
        cs[d] = cv;
        sn[d] = sv;
    }
    __syncthreads();

    const __nv_bfloat16* qrow = p.q + (int64_t)n * p.Hq * D;
    __nv_bfloat16* qdst = p.q_rot + (int64_t)n * p.Hq * D;
    const __nv_bfloat16* krow = p.k_new + (int64_t)n * p.Hkv * D;
    const __nv_bfloat16* vrow = p.v_new + (int64_t)n * p.Hkv * D;
    if ((half & 7) == 0) {
        // 16-byte groups: group g < half/8 rotates with group g + half/8;
        // groups from R/8 on are copied
        const int rot = half / 8, copy = (D - p.R) / 8, per_head = rot + copy;
        for (int idx = threadIdx.x; idx < (p.Hq + p.Hkv) * per_head; idx += blockDim.x) {
            const int h = idx / per_head, gidx = idx % per_head;
            const bool is_q = h < p.Hq;
            const int hh = is_q ? h : h - p.Hq;
            const __nv_bfloat16* src = is_q ? qrow + hh * D : krow + hh * D;
            __nv_bfloat16* dst = is_q ? qdst + hh * D : p.K + ((int64_t)hh * p.slab_rows + slot) * D;
            if (gidx < rot) {
                const int d0 = gidx * 8;
                uint4 a = *reinterpret_cast<const uint4*>(src + d0);
                uint4 bb = *reinterpret_cast<const uint4*>(src + d0 + half);
                rotate8(a, bb, cs, sn, d0);
                *reinterpret_cast<uint4*>(dst + d0) = a;
                *reinterpret_cast<uint4*>(dst + d0 + half) = bb;
            } else {
                const int d0 = p.R + (gidx - rot) * 8;
                *reinterpret_cast<uint4*>(dst + d0) = *reinterpret_cast<const uint4*>(src + d0);
            }
        }
        for (int idx = threadIdx.x; idx < p.Hkv * (D / 8); idx += blockDim.x) {
            const int h = idx / (D / 8), d0 = (idx % (D / 8)) * 8;
            *reinterpret_cast<uint4*>(p.V + ((int64_t)h * p.slab_rows + slot) * D + d0) =
                *reinterpret_cast<const uint4*>(vrow + h * D + d0);
        }
    } else {
        auto rotated = [&](const __nv_bfloat16* row, int d) -> float {
            const float x = __bfloat162float(row[d]);
            if (d >= p.R) return x;
            if (d < half) return x * cs[d] - __bfloat162float(row[d + half]) * sn[d];
            return x * cs[d - half] + __bfloat162float(row[d - half]) * sn[d - half];
        };
        for (int idx = threadIdx.x; idx < p.Hq * D; idx += blockDim.x)
            qdst[idx] = __float2bfloat16_rn(rotated(qrow + (idx / D) * D, idx % D));
        for (int idx = threadIdx.x; idx < p.Hkv * D; idx += blockDim.x) {
            const int h = idx / D, d = idx % D;
            const int64_t dst = ((int64_t)h * p.slab_rows + slot) * D + d;
            p.K[dst] = __float2bfloat16_rn(rotated(krow + h * D, d));
            p.V[dst] = vrow[h * D + d];
        }
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

// grid (tiles, kRows / 8): one warp per query row, lanes over head_dim.
__global__ void __launch_bounds__(256) attn_combine_kernel(const __grid_constant__ AttnParams p) {
    const int tile = blockIdx.x;
    const int r = blockIdx.y * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    int b, kvh, qt, sp;
    decode_item(p, tile * p.n_split, b, kvh, qt, sp);
    const AttnChar& c = p.ch[b];
    const int tok = qt * p.tok_per_tile + r / p.g;
    if (tok >= c.M) return;
    const int D = p.D;
    const int64_t item0 = (int64_t)tile * p.n_split;
    float ms[16], ws[16];
    float mx = -INFINITY;
    for (int s = 0; s < p.n_split; ++s) {
        ms[s] = p.part_ml[((item0 + s) * kRows + r) * 2];
        mx = fmaxf(mx, ms[s]);
    }
    float den = 0.f;
    for (int s = 0; s < p.n_split; ++s) {
        ws[s] = (ms[s] == -INFINITY) ? 0.f : exp2f(ms[s] - mx);
        den += ws[s] * p.part_ml[((item0 + s) * kRows + r) * 2 + 1];
    }
    const float inv = 1.f / den;
    const int hq = kvh * p.g + (r % p.g);
    __nv_bfloat16* o = p.out + ((int64_t)(c.tail_off + tok) * p.Hq + hq) * D;
    for (int v4 = lane; v4 < D / 4; v4 += 32) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s = 0; s < p.n_split; ++s) {
            if (ws[s] == 0.f) continue;
            const float4 x = *reinterpret_cast<const float4*>(p.part_o + ((item0 + s) * kRows + r) * D + v4 * 4);
            acc.x += ws[s] * x.x; acc.y += ws[s] * x.y; acc.z += ws[s] * x.z; acc.w += ws[s] * x.w;
        }
        const uint2 packed = make_uint2(f2_to_bf2(acc.x * inv, acc.y * inv), f2_to_bf2(acc.z * inv, acc.w * inv));
        *reinterpret_cast<uint2*>(o + v4 * 4) = packed;
    }
}

}  // namespace

void launch_rope_append(const AttnParams& p, int total_tokens, cudaStream_t s) {
    if (total_tokens <= 0) return;
    rope_append_kernel<<<total_tokens, 128, 0, s>>>(p);
}

void launch_attn_combine(const AttnParams& p, int n_tiles, cudaStream_t s) {
    if (n_tiles <= 0 || p.n_split <= 1) return;
    attn_combine_kernel<<<dim3(n_tiles, kRows / 8), 256, 0, s>>>(p);
}

}  // namespace kvm
