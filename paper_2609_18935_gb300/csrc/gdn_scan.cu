// Gated delta rule from the carried state (Eq. 3 for a recurrent layer;
// recurrence of Gated DeltaNet, the layer family named in §4.1):
//     S_t = alpha_t S_{t-1} (I - beta_t k_t k_t^T) + beta_t v_t k_t^T,  o_t = S_t q_t.
//
// Chunked (WY/UT) evaluation, chunks of C = 64 tokens starting at the first
// tail token.  For a chunk from state S0, with g_t = sum_{u<=t} log alpha_u:
//   L[t][j] = exp(g_t - g_j) beta_j (k_t . k_j), j < t       (strictly lower)
//   (I + L) U = V,  (I + L) W = diag(exp g) K                 (forward substitution)
//   E = U - W S0^T
//   O = diag(exp g) Q S0^T + A E,  A[t][j] = exp(g_t - g_j) beta_j (q_t . k_j), j <= t
//   S = exp(g_last) S0 + E^T diag(beta_j exp(g_last - g_j)) K
// Rows of S evolve independently, so a block owns 32 rows (d_v tile) of one
// head of one character and carries them through every chunk in order.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

constexpr int C = 64;          // chunk length
constexpr int DVT = 32;        // rows of S per block
constexpr int kThreads = 256;

template <int DK>
struct Smem {
    static constexpr int KP = DK + 1;
    static constexpr int floats = 3 * C * KP /*K,Q,W*/ + C * (DVT + 1) /*V/U/E*/ + DVT * KP /*S*/ +
                                  2 * C * (C + 1) /*L, A*/ + 3 * C /*g, beta, wS*/;
};

template <int DK>
__global__ void __launch_bounds__(kThreads) gdn_chunk_scan_kernel(const __grid_constant__ GdnParams p) {
    constexpr int KP = DK + 1;
    extern __shared__ float sm[];
    float* Ks = sm;                       // [C][KP]
    float* Qs = Ks + C * KP;              // [C][KP]
    float* Ws = Qs + C * KP;              // [C][KP]   exp(g) K, solved in place into W
    float* Vs = Ws + C * KP;              // [C][DVT+1] V, solved in place into U, then E
    float* Ss = Vs + C * (DVT + 1);       // [DVT][KP]  state rows r0 .. r0+31
    float* Lm = Ss + DVT * KP;            // [C][C+1]
    float* Am = Lm + C * (C + 1);         // [C][C+1]
    float* gs = Am + C * (C + 1);         // [C]
    float* bs = gs + C;                   // [C]
    float* ws = bs + C;                   // [C]  beta_j exp(g_last - g_j)

    const int tid = threadIdx.x;
    const int r0 = blockIdx.x * DVT;
    const int h = blockIdx.y;
    const int b = blockIdx.z;
    const GdnChar ch = p.ch[b];
    if (ch.M <= 0) return;
    const int H = p.H, dv = p.dv;
    float* Sg = p.S + (((int64_t)b * H + h) * dv + r0) * DK;

    for (int idx = tid; idx < DVT * DK; idx += kThreads)
        Ss[(idx / DK) * KP + idx % DK] = Sg[idx];

    for (int c0 = 0; c0 < ch.M; c0 += C) {
        const int n = min(C, ch.M - c0);
        const int64_t tok0 = ch.tail_off + c0;
        __syncthreads();
        // ---- load the chunk (rows >= n are zero)
        for (int idx = tid; idx < C * DK; idx += kThreads) {
            const int t = idx / DK, cc = idx % DK;
            float kv = 0.f, qv = 0.f;
            if (t < n) {
                const int64_t off = ((tok0 + t) * H + h) * DK + cc;
                kv = __bfloat162float(p.k[off]);
                qv = __bfloat162float(p.q[off]);
            }
            Ks[t * KP + cc] = kv;
            Qs[t * KP + cc] = qv;
        }
        for (int idx = tid; idx < C * DVT; idx += kThreads) {
            const int t = idx / DVT, r = idx % DVT;
            Vs[t * (DVT + 1) + r] = t < n ? __bfloat162float(p.v[((tok0 + t) * H + h) * dv + r0 + r]) : 0.f;
        }
        if (tid < 32) {
            // inclusive prefix sums of log alpha over the chunk (two 32-token halves)
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
        __syncthreads();
        const float g_last = gs[n - 1];
        if (tid < C) ws[tid] = tid < n ? bs[tid] * expf(g_last - gs[tid]) : 0.f;
        // ---- L and A (64 x 64), W init
        for (int e = tid; e < C * C; e += kThreads) {
            const int t = e / C, j = e % C;
            float dkk = 0.f, dqk = 0.f;
            if (j <= t && t < n) {
#pragma unroll 8
                for (int cc = 0; cc < DK; ++cc) {
                    const float kj = Ks[j * KP + cc];
                    dkk = fmaf(Ks[t * KP + cc], kj, dkk);
                    dqk = fmaf(Qs[t * KP + cc], kj, dqk);
                }
            }
            const float dec = (j <= t && t < n) ? expf(gs[t] - gs[j]) * bs[j] : 0.f;
            Lm[t * (C + 1) + j] = j < t ? dec * dkk : 0.f;
            Am[t * (C + 1) + j] = dec * dqk;
        }
        for (int idx = tid; idx < C * DK; idx += kThreads) {
            const int t = idx / DK, cc = idx % DK;
            Ws[t * KP + cc] = t < n ? expf(gs[t]) * Ks[t * KP + cc] : 0.f;
        }
        __syncthreads();
        // ---- forward substitution: one column of [V | exp(g) K] per thread
        if (tid < DVT + DK) {
            float* col = tid < DVT ? (Vs + tid) : (Ws + (tid - DVT));
            const int stride = tid < DVT ? (DVT + 1) : KP;
            for (int t = 1; t < n; ++t) {
                float acc = col[t * stride];
                for (int j = 0; j < t; ++j) acc = fmaf(-Lm[t * (C + 1) + j], col[j * stride], acc);
                col[t * stride] = acc;
            }
        }
        __syncthreads();
        // ---- E = U - W S0^T   (64 x 32, 8 per thread)
        {
            float ev[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int e = tid + k * kThreads;
                const int t = e / DVT, r = e % DVT;
                float acc = 0.f;
#pragma unroll 8
                for (int cc = 0; cc < DK; ++cc) acc = fmaf(Ws[t * KP + cc], Ss[r * KP + cc], acc);
                ev[k] = Vs[t * (DVT + 1) + r] - acc;
            }
            __syncthreads();
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int e = tid + k * kThreads;
                Vs[(e / DVT) * (DVT + 1) + e % DVT] = (e / DVT) < n ? ev[k] : 0.f;
            }
        }
        __syncthreads();
        // ---- O = diag(exp g) Q S0^T + A E
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int e = tid + k * kThreads;
            const int t = e / DVT, r = e % DVT;
            if (t >= n) continue;
            float qs = 0.f;
#pragma unroll 8
            for (int cc = 0; cc < DK; ++cc) qs = fmaf(Qs[t * KP + cc], Ss[r * KP + cc], qs);
            float ae = 0.f;
            for (int j = 0; j <= t; ++j) ae = fmaf(Am[t * (C + 1) + j], Vs[j * (DVT + 1) + r], ae);
            const float o = expf(gs[t]) * qs + ae;
            p.out[((tok0 + t) * H + h) * dv + r0 + r] = __float2bfloat16_rn(o);
        }
        __syncthreads();
        // ---- S = exp(g_last) S0 + E^T diag(ws) K
        {
            const float gl = expf(g_last);
            for (int e = tid; e < DVT * DK; e += kThreads) {
                const int r = e / DK, cc = e % DK;
                float acc = 0.f;
                for (int j = 0; j < n; ++j) acc = fmaf(Vs[j * (DVT + 1) + r] * ws[j], Ks[j * KP + cc], acc);
                Ss[r * KP + cc] = gl * Ss[r * KP + cc] + acc;
            }
        }
    }
    __syncthreads();
    for (int idx = tid; idx < DVT * DK; idx += kThreads)
        Sg[idx] = Ss[(idx / DK) * KP + idx % DK];
}

template <int DK>
void launch_dk(const GdnParams& p, cudaStream_t s) {
    const size_t smem = sizeof(float) * Smem<DK>::floats;
    static unsigned long long configured = 0;   // one bit per device
    int dev = 0;
    cudaGetDevice(&dev);
    if (!(configured >> (dev & 63) & 1ull)) {
        cudaFuncSetAttribute(gdn_chunk_scan_kernel<DK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        configured |= 1ull << (dev & 63);
    }
    dim3 grid(p.dv / DVT, p.H, p.n_chars);
    gdn_chunk_scan_kernel<DK><<<grid, kThreads, smem, s>>>(p);
}

}  // namespace

void launch_gdn_chunk_scan(const GdnParams& p, cudaStream_t s) {
    if (p.dk == 64) launch_dk<64>(p, s);
    else if (p.dk == 128) launch_dk<128>(p, s);
}

}  // namespace kvm
