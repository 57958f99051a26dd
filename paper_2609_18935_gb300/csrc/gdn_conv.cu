// Short convolution of a gated-delta-rule layer with its carried state (the
// convolution part of R_t, §4.1: it continues across rounds without rollback,
// like S).  Each channel c of the layer's q, k and v projections (channels
// ordered q [H][d_k], k [H][d_k], v [H][d_v]) is filtered by a causal
// depthwise convolution of width 4 and passed through SiLU:
//     y_t[c] = silu(sum_{i=0..3} w[c][i] x_{t-3+i}[c]),
// where x_{-3..-1} are the last three inputs of earlier rounds (the conv
// state; zero for a fresh context).  Each head's k is then scaled to unit L2
// norm (the delta rule's keys); q and v are not.  The outputs are rounded to
// bf16, the delta rule's operand type.
//
// grid.x < sum M: one block per (tail token, head) computes y for its head's
// q, k and v channels; grid.x >= sum M: one block per (character, head)
// writes the character's new state (the last three inputs of [state; tail])
// into the other of two state buffers, so that no block reads a state row
// that another block of the same launch writes.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

__device__ __forceinline__ float silu(float x) { return x / (1.f + __expf(-x)); }

// First channel of the k part (q channels come first, then k, then v).
__device__ __forceinline__ int H_off_k(const ConvParams& p) { return p.H * p.dk; }

__global__ void __launch_bounds__(128) gdn_conv_kernel(const __grid_constant__ ConvParams p) {
    grid_dependency_wait();
    grid_dependents_launch();
    const int h = blockIdx.y;
    const int dk = p.dk, dv = p.dv, C = p.channels;
    const int per_head = 2 * dk + dv;
    if ((int)blockIdx.x >= p.total) {
        // new conv state of one character's channels of head h
        const int b = blockIdx.x - p.total;
        if (b >= p.n_chars) { if (threadIdx.x == 0) atomicOr(p.err, kErrBounds); return; }
        const int M = p.tail_cu[b + 1] - p.tail_cu[b];
        const __nv_bfloat16* old_s = p.state_in + (int64_t)b * 3 * C;
        __nv_bfloat16* new_s = p.state_out + (int64_t)b * 3 * C;
        for (int e = threadIdx.x; e < 3 * per_head; e += blockDim.x) {
            const int r = e / per_head, j = e % per_head;
            // channel of element j of this head
            const int c = j < dk ? h * dk + j
                        : j < 2 * dk ? H_off_k(p) + h * dk + (j - dk) : 2 * H_off_k(p) + h * dv + (j - 2 * dk);
            const int t = M - 3 + r;                         // position in the tail (negative: old state row t + 3)
            __nv_bfloat16 x;
            if (t >= 0) {
                const int64_t tok = p.tail_cu[b] + t;
                x = j < dk ? p.xq[(tok * p.H + h) * dk + j]
                  : j < 2 * dk ? p.xk[(tok * p.H + h) * dk + (j - dk)]
                               : p.xv[(tok * p.H + h) * dv + (j - 2 * dk)];
            } else {
                x = old_s[(int64_t)(t + 3) * C + c];
            }
            new_s[(int64_t)r * C + c] = x;
        }
        return;
    }
    const int n = blockIdx.x;                                // packed tail token
    int lo = 0, hi = p.n_chars - 1;                          // last b with tail_cu[b] <= n
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.tail_cu[mid] <= n) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const int t = n - p.tail_cu[b];
    const __nv_bfloat16* old_s = p.state_in + (int64_t)b * 3 * C;
    __shared__ float ksq[4];
    float kval = 0.f;                                        // d_k <= 128 threads: at most one k channel each
    float part = 0.f;
    for (int j = threadIdx.x; j < per_head; j += blockDim.x) {
        const bool is_q = j < dk, is_k = !is_q && j < 2 * dk;
        const int jj = is_q ? j : is_k ? j - dk : j - 2 * dk;
        const int c = is_q ? h * dk + jj : is_k ? H_off_k(p) + h * dk + jj : 2 * H_off_k(p) + h * dv + jj;
        const __nv_bfloat16* src = is_q ? p.xq : is_k ? p.xk : p.xv;
        const int width = (is_q || is_k) ? dk : dv;
        float acc = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int tt = t - 3 + i;                         // input row of tap i
            float x;
            if (tt >= 0) x = __bfloat162float(src[((int64_t)(p.tail_cu[b] + tt) * p.H + h) * width + jj]);
            else x = __bfloat162float(old_s[(int64_t)(tt + 3) * C + c]);
            acc = fmaf(p.w[(int64_t)c * 4 + i], x, acc);
        }
        const float y = silu(acc);
        if (is_k) {
            kval = y;                                         // normalised below
            part = fmaf(y, y, part);
        } else {
            __nv_bfloat16* dst = is_q ? p.yq : p.yv;
            dst[((int64_t)n * p.H + h) * width + jj] = __float2bfloat16_rn(y);
        }
    }
    // ||k||^2 over the head: warp sums, then the block's four warps
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if ((threadIdx.x & 31) == 0) ksq[threadIdx.x >> 5] = part;
    __syncthreads();
    const float norm2 = ksq[0] + ksq[1] + ksq[2] + ksq[3];
    const float inv = norm2 > 0.f ? rsqrtf(norm2) : 0.f;
    for (int j = threadIdx.x; j < per_head; j += blockDim.x)
        if (j >= dk && j < 2 * dk) p.yk[((int64_t)n * p.H + h) * dk + (j - dk)] = __float2bfloat16_rn(kval * inv);
}

}  // namespace

void launch_gdn_conv(const ConvParams& p, cudaStream_t s) {
    if (p.total <= 0) return;
    launch_pdl(gdn_conv_kernel, dim3(p.total + p.n_chars, p.H), dim3(128), 0, s, p);
}

}  // namespace kvm
