// Attention-probe diagnostics (§5.3; Appendix C): the attention distribution
// of a character's last n_q query tokens over its live KV, reconstructed with
// a float32 reference softmax and averaged over those queries and every query
// head of one attention layer.  Removed records left holes in position space
// only: the compacted cache holds live entries alone, so the softmax
// denominator runs over live tokens (holes excluded) by construction.
//
// Query i of the probe (0 <= i < n_q) is the live entry L - n_q + i; it sees
// live entries 0 .. L - n_q + i (causal in processing order), with scores
// q_i . k_j / sqrt(D) in fp32, q_i rotated at that entry's position.
//
//  probe_rotate : rotate the caller's probe queries (fp64 angle reduced mod
//                 2 pi, fp32 rotation) into an fp32 workspace;
//  probe_tiles  : (pass A) per 64-key tile and query row, the tile's max
//                 score and sum of exp(s - max);
//  probe_rows   : per query row, the softmax max and denominator from the
//                 tiles' partials;
//  probe_tiles  : (pass C) the scores again, p = exp(s - max) / sum, summed
//                 over every query row: the averaged distribution of each
//                 key, and its group's mass (atomic adds) when groups are
//                 given.
// This is a diagnostic, not the hot path: fp32 on the CUDA cores, scores
// recomputed in pass C rather than stored.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

constexpr double kTwoPiP = 6.283185307179586476925286766559;
constexpr int kProbeThreads = 256;
constexpr int kRowChunk = 64;                  // query rows staged per step
constexpr int kRowsPerThread = kRowChunk / (kProbeThreads / kProbeKeys);   // 16

__global__ void __launch_bounds__(128) probe_rotate_kernel(const __grid_constant__ ProbeParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int i = blockIdx.x;
    const int64_t pos = p.pos[p.slot0 + p.L - p.n_q + i];
    const int half = p.R / 2;
    __shared__ float cs[kMaxRotaryHalf], sn[kMaxRotaryHalf];
    for (int d = threadIdx.x; d < half; d += blockDim.x) {
        const double ang = (double)pos * p.inv_freq[d];
        const double r = fma(-rint(ang * (1.0 / kTwoPiP)), kTwoPiP, ang);
        float sv, cv;
        sincosf((float)r, &sv, &cv);
        cs[d] = cv;
        sn[d] = sv;
    }
    __syncthreads();
    const __nv_bfloat16* q = p.q + (int64_t)i * p.Hq * p.D;
    float* o = p.q_rot + (int64_t)i * p.Hq * p.D;
    for (int idx = threadIdx.x; idx < p.Hq * p.D; idx += blockDim.x) {
        const int d = idx % p.D, row = idx - d;
        const float x = __bfloat162float(q[idx]);
        float y = x;
        if (d < half) y = x * cs[d] - __bfloat162float(q[row + d + half]) * sn[d];
        else if (d < p.R) y = x * cs[d - half] + __bfloat162float(q[row + d - half]) * sn[d - half];
        o[idx] = y;
    }
}

// Shared memory: the key tile of one KV head [64][D + 2] bf16 (the pad makes
// the row stride an odd number of words, so lanes reading different keys at
// the same column hit different banks), then a chunk of query rows
// [64][D] fp32 (read as broadcasts), then the reduction scratch.
template <bool kFinal>
__global__ void __launch_bounds__(kProbeThreads) probe_tiles_kernel(const __grid_constant__ ProbeParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    extern __shared__ __align__(16) uint8_t smem[];
    const int D = p.D, KS = D / 2 + 1;                     // key row stride in 32-bit words
    uint32_t* Ks = reinterpret_cast<uint32_t*>(smem);
    float* Qs = reinterpret_cast<float*>(smem + (size_t)kProbeKeys * KS * 4);
    float* red = Qs + (size_t)kRowChunk * D;                // [rsub][half][rows][2] = 4 * 2 * 16 * 2
    float* acc_s = red + 4 * 2 * kRowsPerThread * 2;        // [4][64] per-key partial sums (pass C)
    const int t = threadIdx.x;
    const int kk = t & (kProbeKeys - 1), rsub = t / kProbeKeys, whalf = kk >> 5;
    const int tile = blockIdx.x;
    const int j = tile * kProbeKeys + kk;                   // this thread's key (live index)
    const int rows_kv = p.n_q * p.g;
    const int n_rows = p.n_q * p.Hq;
    const int first_q = p.L - p.n_q;                        // live index of probe query 0
    float acc = 0.f;

    for (int kv = 0; kv < p.Hkv; ++kv) {
        __syncthreads();                                    // the previous key tile is consumed
        const __nv_bfloat16* kb = p.K + ((int64_t)kv * p.slab_rows + p.slot0 + (int64_t)tile * kProbeKeys) * D;
        for (int idx = t; idx < kProbeKeys * (D / 2); idx += kProbeThreads) {
            const int r = idx / (D / 2), w = idx % (D / 2);
            const bool in = tile * kProbeKeys + r < p.L;
            Ks[r * KS + w] = in ? reinterpret_cast<const uint32_t*>(kb + (int64_t)r * D)[w] : 0u;
        }
        for (int c0 = 0; c0 < rows_kv; c0 += kRowChunk) {
            __syncthreads();                                // the previous query chunk is consumed
            for (int idx = t; idx < kRowChunk * D; idx += kProbeThreads) {
                const int r = idx / D, d = idx % D, rg = c0 + r;
                float v = 0.f;
                if (rg < rows_kv) {
                    const int i = rg / p.g, h = kv * p.g + rg % p.g;
                    v = p.q_rot[((int64_t)i * p.Hq + h) * D + d];
                }
                Qs[idx] = v;
            }
            __syncthreads();
            float s[kRowsPerThread];
#pragma unroll
            for (int r = 0; r < kRowsPerThread; ++r) s[r] = 0.f;
            const uint32_t* krow = Ks + kk * KS;
            const float* qb = Qs + (size_t)(rsub * kRowsPerThread) * D;
            for (int w = 0; w < D / 2; ++w) {
                const uint32_t kw = krow[w];
                const float k0 = __uint_as_float(kw << 16), k1 = __uint_as_float(kw & 0xffff0000u);
#pragma unroll
                for (int r = 0; r < kRowsPerThread; ++r) {
                    const float2 q2 = *reinterpret_cast<const float2*>(qb + (size_t)r * D + 2 * w);
                    s[r] = fmaf(q2.x, k0, fmaf(q2.y, k1, s[r]));
                }
            }
            // mask: rows past the end, keys past the row's causal limit
#pragma unroll
            for (int r = 0; r < kRowsPerThread; ++r) {
                const int rg = c0 + rsub * kRowsPerThread + r;
                const int i = rg / p.g;
                const bool vis = rg < rows_kv && j < p.L && j <= first_q + i;
                s[r] = vis ? s[r] * p.scale : -INFINITY;
            }
            if (!kFinal) {
                // per row: this warp's (max, sum over its 32 keys), then the
                // two warps of the row group combine
#pragma unroll
                for (int r = 0; r < kRowsPerThread; ++r) {
                    float m = s[r];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                    float e = (m == -INFINITY) ? 0.f : expf(s[r] - m);
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) e += __shfl_xor_sync(0xffffffffu, e, o);
                    if ((t & 31) == 0) {
                        red[((rsub * 2 + whalf) * kRowsPerThread + r) * 2 + 0] = m;
                        red[((rsub * 2 + whalf) * kRowsPerThread + r) * 2 + 1] = e;
                    }
                }
                __syncthreads();
                if (kk < kRowsPerThread) {                  // one thread per (rsub, row)
                    const int r = kk;
                    const int rg = c0 + rsub * kRowsPerThread + r;
                    if (rg < rows_kv) {
                        const float m0 = red[((rsub * 2 + 0) * kRowsPerThread + r) * 2 + 0];
                        const float e0 = red[((rsub * 2 + 0) * kRowsPerThread + r) * 2 + 1];
                        const float m1 = red[((rsub * 2 + 1) * kRowsPerThread + r) * 2 + 0];
                        const float e1 = red[((rsub * 2 + 1) * kRowsPerThread + r) * 2 + 1];
                        const float m = fmaxf(m0, m1);
                        const float e = (m == -INFINITY) ? 0.f : e0 * expf(m0 - m) + e1 * expf(m1 - m);
                        const int row = (rg / p.g) * p.Hq + kv * p.g + rg % p.g;
                        p.part[((int64_t)tile * n_rows + row) * 2 + 0] = m;
                        p.part[((int64_t)tile * n_rows + row) * 2 + 1] = e;
                    }
                }
            } else {
#pragma unroll
                for (int r = 0; r < kRowsPerThread; ++r) {
                    const int rg = c0 + rsub * kRowsPerThread + r;
                    if (rg < rows_kv && s[r] != -INFINITY) {
                        const int row = (rg / p.g) * p.Hq + kv * p.g + rg % p.g;
                        const float m = p.row_ms[2 * row], den = p.row_ms[2 * row + 1];
                        acc += expf(s[r] - m) / den;
                    }
                }
            }
        }
    }
    if (kFinal) {
        acc_s[rsub * kProbeKeys + kk] = acc;
        __syncthreads();
        if (rsub == 0 && j < p.L) {
            const float tot = (acc_s[kk] + acc_s[kProbeKeys + kk] + acc_s[2 * kProbeKeys + kk] +
                               acc_s[3 * kProbeKeys + kk]) / (float)n_rows;
            p.probs[j] = tot;
            if (p.group_of) {
                const int gid = p.group_of[j];
                if (gid >= p.n_groups) atomicOr(p.err, kErrBounds);
                else if (gid >= 0) atomicAdd(p.group_mass + gid, tot);
            }
        }
    }
}

__global__ void probe_rows_kernel(const __grid_constant__ ProbeParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int row = blockIdx.x * blockDim.x + threadIdx.x;
    const int n_rows = p.n_q * p.Hq;
    if (row >= n_rows) return;
    const int tiles = (p.L + kProbeKeys - 1) / kProbeKeys;
    float m = -INFINITY, e = 0.f;
    for (int tl = 0; tl < tiles; ++tl) {
        const float mt = p.part[((int64_t)tl * n_rows + row) * 2 + 0];
        const float et = p.part[((int64_t)tl * n_rows + row) * 2 + 1];
        if (mt == -INFINITY) continue;
        const float nm = fmaxf(m, mt);
        e = (m == -INFINITY ? 0.f : e * expf(m - nm)) + et * expf(mt - nm);
        m = nm;
    }
    p.row_ms[2 * row] = m;
    p.row_ms[2 * row + 1] = e;
}

size_t probe_smem(int D) {
    return (size_t)kProbeKeys * (D / 2 + 1) * 4 + (size_t)kRowChunk * D * 4 + 4 * 2 * kRowsPerThread * 2 * 4 +
           4 * kProbeKeys * 4;
}

template <auto KERNEL>
void probe_configure(size_t smem) {
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(KERNEL, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        configured |= 1ull << (dev & 63);
    }
}

}  // namespace

void launch_attn_probe(const ProbeParams& p, cudaStream_t s) {
    if (p.L <= 0 || p.n_q <= 0) return;
    const int tiles = (p.L + kProbeKeys - 1) / kProbeKeys;
    const size_t smem = probe_smem(p.D);
    probe_configure<probe_tiles_kernel<false>>(smem);
    probe_configure<probe_tiles_kernel<true>>(smem);
    launch_pdl(probe_rotate_kernel, dim3(p.n_q), dim3(128), 0, s, p);
    launch_pdl(probe_tiles_kernel<false>, dim3(tiles), dim3(kProbeThreads), smem, s, p);
    launch_pdl(probe_rows_kernel, dim3((p.n_q * p.Hq + 127) / 128), dim3(128), 0, s, p);
    launch_pdl(probe_tiles_kernel<true>, dim3(tiles), dim3(kProbeThreads), smem, s, p);
}

}  // namespace kvm
