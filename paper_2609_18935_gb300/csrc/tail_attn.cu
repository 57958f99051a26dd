// True-tail prefill for one full-attention layer (Eq. 3, §4.2): the kernels
// around the tensor-core attention (tail_attn_tc.cu).
//
//  rope_append : rotate the tail's q and k at positions p + i, append the
//                rotated k and v at live slots L' + i with their positions,
//                and write the rotated q for the attention's Q staging.
//                The angle pos * omega_d is formed and reduced modulo 2*pi in
//                fp64 (positions far beyond the live length stay accurate),
//                then sin/cos and the rotation run in fp32.
//  rerotate    : tail-and-relocate (§5.2): turn stored keys from the
//                positions they were rotated at to new positions, i.e. rotate
//                each rotary pair by (new - old) * omega_d (rotations of a
//                pair compose by adding angles), and relabel the positions.
//  attn_combine : merge the partials of query tiles that the attention's
//                persistent blocks split between them: each partial is an
//                unnormalised accumulator with (reference max in log2 units,
//                sum); a thread per 4-column piece of a row, or per 32-column
//                group when the round shares more tiles than one wave of
//                pieces covers.
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
    grid_dependency_wait();
    grid_dependents_launch();
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
    const int64_t pos = p.tail_pos ? (int64_t)p.tail_pos[n] : c.p + i;
    const int64_t slot = c.cap_off + c.L_prev + i;
    const int half = p.R / 2;
    const int D = p.D;

    __shared__ float cs[kMaxRotaryHalf], sn[kMaxRotaryHalf];
    const __nv_bfloat16* qrow = p.q + (int64_t)n * p.Hq * D;
    __nv_bfloat16* qdst = p.q_rot + (int64_t)n * p.Hq * D;
    const __nv_bfloat16* krow = p.k_new + (int64_t)n * p.Hkv * D;
    const __nv_bfloat16* vrow = p.v_new + (int64_t)n * p.Hkv * D;
    if ((half & 7) == 0) {
        // 16-byte groups: group g < half/8 rotates with group g + half/8;
        // groups from R/8 on are copied.  The first kPre items of each thread
        // are loaded before the angles are formed, so the loads overlap the
        // trigonometry.
        const int rot = half / 8, copy = (D - p.R) / 8, per_head = rot + copy;
        const int n_items = (p.Hq + p.Hkv) * per_head;
        constexpr int kPre = 4;
        auto src_of = [&](int idx, int& d0, bool& rotated, __nv_bfloat16*& dst) -> const __nv_bfloat16* {
            const int h = idx / per_head, gidx = idx % per_head;
            const bool is_q = h < p.Hq;
            const int hh = is_q ? h : h - p.Hq;
            dst = is_q ? qdst + hh * D : p.K + ((int64_t)hh * p.slab_rows + slot) * D;
            rotated = gidx < rot;
            d0 = rotated ? gidx * 8 : p.R + (gidx - rot) * 8;
            return is_q ? qrow + hh * D : krow + hh * D;
        };
        uint4 la[kPre], lb[kPre];
#pragma unroll
        for (int u = 0; u < kPre; ++u) {
            const int idx = threadIdx.x + u * blockDim.x;
            if (idx < n_items) {
                int d0; bool rotated; __nv_bfloat16* dst;
                const __nv_bfloat16* src = src_of(idx, d0, rotated, dst);
                la[u] = *reinterpret_cast<const uint4*>(src + d0);
                if (rotated) lb[u] = *reinterpret_cast<const uint4*>(src + d0 + half);
            }
        }
        // v needs no angle: copy it first, from the block's last threads, so
        // that the first ones form the angles meanwhile
        for (int idx = blockDim.x - 1 - threadIdx.x; idx < p.Hkv * (D / 8); idx += blockDim.x) {
            const int h = idx / (D / 8), d0 = (idx % (D / 8)) * 8;
            *reinterpret_cast<uint4*>(p.V + ((int64_t)h * p.slab_rows + slot) * D + d0) =
                *reinterpret_cast<const uint4*>(vrow + h * D + d0);
        }
        for (int d = threadIdx.x; d < half; d += blockDim.x) {
            const double ang = (double)pos * p.inv_freq[d];
            const double r = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);   // ang mod 2*pi, |r| <= pi
            float sv, cv;
            sincosf((float)r, &sv, &cv);
            cs[d] = cv;
            sn[d] = sv;
        }
        __syncthreads();
#pragma unroll
        for (int u = 0; u < kPre; ++u) {
            const int idx = threadIdx.x + u * blockDim.x;
            if (idx < n_items) {
                int d0; bool rotated; __nv_bfloat16* dst;
                src_of(idx, d0, rotated, dst);
                if (rotated) {
                    rotate8(la[u], lb[u], cs, sn, d0);
                    *reinterpret_cast<uint4*>(dst + d0) = la[u];
                    *reinterpret_cast<uint4*>(dst + d0 + half) = lb[u];
                } else {
                    *reinterpret_cast<uint4*>(dst + d0) = la[u];
                }
            }
        }
        for (int idx = threadIdx.x + kPre * blockDim.x; idx < n_items; idx += blockDim.x) {
            int d0; bool rotated; __nv_bfloat16* dst;
            const __nv_bfloat16* src = src_of(idx, d0, rotated, dst);
            uint4 a = *reinterpret_cast<const uint4*>(src + d0);
            if (rotated) {
                uint4 bb = *reinterpret_cast<const uint4*>(src + d0 + half);
                rotate8(a, bb, cs, sn, d0);
                *reinterpret_cast<uint4*>(dst + d0 + half) = bb;
            }
            *reinterpret_cast<uint4*>(dst + d0) = a;
        }
    } else {
        for (int d = threadIdx.x; d < half; d += blockDim.x) {
            const double ang = (double)pos * p.inv_freq[d];
            const double r = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);
            float sv, cv;
            sincosf((float)r, &sv, &cv);
            cs[d] = cv;
            sn[d] = sv;
        }
        __syncthreads();
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

// grid (n_split_tiles, kRows * D / 4 / 256): the x-th query tile that several
// attention blocks share.  Block cb = split_cb[x] is the first to start
// inside the tile, so its partials are in the slots of blocks c0 = cb - 1 ..
// c1 (the last block that starts inside the tile): c0's last segment (slot
// 2 c0 + 1, or 2 c0 when the tile is also c0's first segment) and the first
// segments 2 c of the others.  A thread owns four columns of one row (rows
// fastest across threads, as in the partial layout) and merges the partials
// online, two at a time, each batch's (max, sum) pairs and O pieces loaded
// together.
// At most 36 registers a thread keep seven blocks on an SM, so that the
// grid of a round with up to 33 shared tiles (x 32 blocks at head_dim 256)
// runs in one wave.
__global__ void __launch_bounds__(256, 7) attn_combine_piece_kernel(const __grid_constant__ AttnParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int cb = p.split_cb[blockIdx.x];
    const int t = p.cta_tile[cb];
    const int c0 = cb - 1;
    int c1 = cb;
    while (c1 + 1 < p.n_ctas && p.cta_tile[c1 + 1] == t && p.cta_k[c1 + 1] > 0) ++c1;
    const int slot0 = (p.cta_tile[c0] == t) ? 2 * c0 : 2 * c0 + 1;
    const int n_parts = c1 - c0 + 1;

    int lo = 0, hi = p.n_chars - 1;                                // last b with tile_off <= t
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].tile_off <= t) lo = mid; else hi = mid - 1;
    }
    const AttnChar& c = p.ch[lo];
    const int local = t - c.tile_off;
    const int kvh = local / c.n_qtiles, qt = local % c.n_qtiles;
    const int D = p.D;
    const int item = blockIdx.y * blockDim.x + threadIdx.x;        // (4-column piece, row): rows fastest
    const int r = item % kRows;
    const int piece = item / kRows;
    if (piece >= D / 4) return;
    const int cg = piece >> 3, q4 = piece & 7;
    const int tok = qt * p.tok_per_tile + r / p.g;
    if (tok >= c.M) return;
    __nv_bfloat16* o = p.out + ((int64_t)(c.tail_off + tok) * p.Hq + kvh * p.g + (r % p.g)) * D + cg * 32 + q4 * 4;
    // this thread's piece of slot s: po + s * D * kRows floats; its (max, sum): pm + s * 2 kRows
    const float* po = p.part_o + ((cg * 8 + q4) * kRows + r) * 4;
    const float* pm = p.part_ml + r * 2;
    const int sstride = D * kRows;
    constexpr int kBatch = 2;
    float mx = -INFINITY, den = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int q0 = 0; q0 < n_parts; q0 += kBatch) {
        float2 ml[kBatch];
        float4 x[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            if (q0 + u < n_parts) {
                const int slot = (q0 + u == 0) ? slot0 : 2 * (c0 + q0 + u);
                ml[u] = *reinterpret_cast<const float2*>(pm + slot * (2 * kRows));
                x[u] = *reinterpret_cast<const float4*>(po + slot * sstride);
            } else {
                ml[u] = make_float2(-INFINITY, 0.f);
            }
        }
        float bm = -INFINITY;
#pragma unroll
        for (int u = 0; u < kBatch; ++u) bm = fmaxf(bm, ml[u].x);
        const float nmx = fmaxf(mx, bm);
        if (nmx == -INFINITY) continue;
        const float sc = (mx == -INFINITY) ? 0.f : exp2f(mx - nmx);
        den *= sc;
        acc.x *= sc; acc.y *= sc; acc.z *= sc; acc.w *= sc;
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            if (ml[u].x == -INFINITY) continue;
            const float w = exp2f(ml[u].x - nmx);
            den += w * ml[u].y;
            acc.x += w * x[u].x; acc.y += w * x[u].y; acc.z += w * x[u].z; acc.w += w * x[u].w;
        }
        mx = nmx;
    }
    const float inv = den > 0.f ? 1.f / den : 0.f;
    *reinterpret_cast<uint2*>(o) = make_uint2(f2_to_bf2(acc.x * inv, acc.y * inv), f2_to_bf2(acc.z * inv, acc.w * inv));
}

// grid (n_split_tiles, kRows * D / 32 / kCombineThreads): the x-th query
// tile that several attention blocks share.  Block cb = split_cb[x] is the
// first to start inside the tile, so its partials are in the slots of blocks
// c0 = cb - 1 .. c1 (the last block that starts inside the tile): c0's last
// segment (slot 2 c0 + 1, or 2 c0 when the tile is also c0's first segment)
// and the first segments 2 c of the others.  A thread owns one 32-column
// group of one row (rows fastest across threads, as in the partial layout)
// and merges the partials online, two at a time: both (max, sum) pairs
// first, then each part's eight 4-column pieces.
constexpr int kCombineThreads = 128;
__global__ void __launch_bounds__(kCombineThreads) attn_combine_group_kernel(const __grid_constant__ AttnParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int cb = p.split_cb[blockIdx.x];
    const int t = p.cta_tile[cb];
    const int c0 = cb - 1;
    int c1 = cb;
    while (c1 + 1 < p.n_ctas && p.cta_tile[c1 + 1] == t && p.cta_k[c1 + 1] > 0) ++c1;
    const int slot0 = (p.cta_tile[c0] == t) ? 2 * c0 : 2 * c0 + 1;
    const int n_parts = c1 - c0 + 1;

    int lo = 0, hi = p.n_chars - 1;                                // last b with tile_off <= t
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].tile_off <= t) lo = mid; else hi = mid - 1;
    }
    const AttnChar& c = p.ch[lo];
    const int local = t - c.tile_off;
    const int kvh = local / c.n_qtiles, qt = local % c.n_qtiles;
    const int D = p.D;
    const int item = blockIdx.y * blockDim.x + threadIdx.x;        // (column group, row): rows fastest
    const int r = item % kRows;
    const int cg = item / kRows;
    if (cg >= D / 32) return;
    const int tok = qt * p.tok_per_tile + r / p.g;
    if (tok >= c.M) return;
    __nv_bfloat16* o = p.out + ((int64_t)(c.tail_off + tok) * p.Hq + kvh * p.g + (r % p.g)) * D + cg * 32;
    // piece q4 of slot s: po + s * D * kRows + q4 * 4 kRows floats; (max, sum): pm + s * 2 kRows
    const float* po = p.part_o + (cg * 8 * kRows + r) * 4;
    const float* pm = p.part_ml + r * 2;
    const int sstride = D * kRows;
    constexpr int kBatch = 2;
    float mx = -INFINITY, den = 0.f;
    float4 acc[8];
#pragma unroll
    for (int q4 = 0; q4 < 8; ++q4) acc[q4] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int q0 = 0; q0 < n_parts; q0 += kBatch) {
        float2 ml[kBatch];
        int slot[kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            slot[u] = (q0 + u == 0) ? slot0 : 2 * (c0 + q0 + u);
            ml[u] = (q0 + u < n_parts) ? *reinterpret_cast<const float2*>(pm + slot[u] * (2 * kRows))
                                       : make_float2(-INFINITY, 0.f);
        }
        float bm = -INFINITY;
#pragma unroll
        for (int u = 0; u < kBatch; ++u) bm = fmaxf(bm, ml[u].x);
        const float nmx = fmaxf(mx, bm);
        if (nmx == -INFINITY) continue;
        const float sc = (mx == -INFINITY) ? 0.f : exp2f(mx - nmx);
        den *= sc;
#pragma unroll
        for (int q4 = 0; q4 < 8; ++q4) {
            acc[q4].x *= sc; acc[q4].y *= sc; acc[q4].z *= sc; acc[q4].w *= sc;
        }
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
            if (ml[u].x == -INFINITY) continue;
            const float w = exp2f(ml[u].x - nmx);
            den += w * ml[u].y;
            const float* src = po + slot[u] * sstride;
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
                const float4 x = *reinterpret_cast<const float4*>(src + q4 * 4 * kRows);
                acc[q4].x += w * x.x; acc[q4].y += w * x.y; acc[q4].z += w * x.z; acc[q4].w += w * x.w;
            }
        }
        mx = nmx;
    }
    const float inv = den > 0.f ? 1.f / den : 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e)
        reinterpret_cast<uint4*>(o)[e] = make_uint4(f2_to_bf2(acc[2 * e].x * inv, acc[2 * e].y * inv),
                                                    f2_to_bf2(acc[2 * e].z * inv, acc[2 * e].w * inv),
                                                    f2_to_bf2(acc[2 * e + 1].x * inv, acc[2 * e + 1].y * inv),
                                                    f2_to_bf2(acc[2 * e + 1].z * inv, acc[2 * e + 1].w * inv));
}

// One block per entry; a thread rotates 2-element pairs (d, d + R/2) of one
// (layer, KV head) key, with the entry's angles formed once in shared memory.
__global__ void __launch_bounds__(256) rerotate_kernel(const __grid_constant__ RerotateParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int j = blockIdx.x;
    if (j >= p.n) return;
    const int64_t slot = p.slot0 + j;
    const int half = p.R / 2;
    __shared__ float cs[kMaxRotaryHalf], sn[kMaxRotaryHalf];
    const int64_t delta = (int64_t)p.new_pos[j] - (int64_t)p.pos[slot];
    for (int d = threadIdx.x; d < half; d += blockDim.x) {
        const double ang = (double)delta * p.inv_freq[d];
        const double r = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);   // ang mod 2*pi, |r| <= pi
        float sv, cv;
        sincosf((float)r, &sv, &cv);
        cs[d] = cv;
        sn[d] = sv;
    }
    __syncthreads();
    const int n_items = p.n_attn * p.Hkv * half;
    for (int idx = threadIdx.x; idx < n_items; idx += blockDim.x) {
        const int d = idx % half, kh = idx / half;          // kh = layer * Hkv + head
        __nv_bfloat16* row = p.K + ((int64_t)kh * p.slab_rows + slot) * p.D;
        const float x = __bfloat162float(row[d]), y = __bfloat162float(row[d + half]);
        row[d] = __float2bfloat16_rn(x * cs[d] - y * sn[d]);
        row[d + half] = __float2bfloat16_rn(y * cs[d] + x * sn[d]);
    }
    __syncthreads();                                        // every thread has read pos[slot]
    if (threadIdx.x == 0) p.pos[slot] = p.new_pos[j];
}

}  // namespace

void launch_rerotate(const RerotateParams& p, cudaStream_t s) {
    if (p.n <= 0) return;
    launch_pdl(rerotate_kernel, dim3(p.n), dim3(256), 0, s, p);
}

void launch_rope_append(const AttnParams& p, int total_tokens, cudaStream_t s) {
    if (total_tokens <= 0) return;
    launch_pdl(rope_append_kernel, dim3(total_tokens), dim3(128), 0, s, p);
}

void launch_attn_combine(const AttnParams& p, cudaStream_t s) {
    if (p.n_split_tiles <= 0) return;
    // one 4-column piece a thread while that grid is one wave (seven blocks
    // an SM), else a 32-column group a thread: at npc (32 shared tiles) the
    // piece form took 11.0 against 12.4 us, at long (128) 16.3 against 13.1
    static int sms_of[64] = {};                      // per device
    int dev = 0;
    cudaGetDevice(&dev);
    int& sms = sms_of[dev & 63];
    if (!sms) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int piece_blocks = (kRows * (p.D / 4) + 255) / 256;
    if ((int64_t)p.n_split_tiles * piece_blocks <= 7 * (int64_t)sms)
        launch_pdl(attn_combine_piece_kernel, dim3(p.n_split_tiles, piece_blocks), dim3(256), 0, s, p);
    else
        launch_pdl(attn_combine_group_kernel, dim3(p.n_split_tiles, (kRows * (p.D / 32) + kCombineThreads - 1) / kCombineThreads),
                   dim3(kCombineThreads), 0, s, p);
}

}  // namespace kvm
