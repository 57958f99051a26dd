// KV removal by in-place compaction (Eq. 2: A_bar = A \ A[D_t]).
//
// Every (attention layer, KV head, K|V) slab of a character, and the
// character's position slab, lose the same live indices.  A survivor at old
// index i moves to i - (removed indices below i); survivors before the first
// removed index stay where they are, so only the suffix moves.
//
// One pass, in place, each moved byte read once and written once:
//   * a slab's moved destination rows [first, L') are cut into chunks of
//     `rows` rows; a block takes chunks of its slab in ticket order;
//   * the block loads all of its chunk's source rows into registers, then
//     publishes a per-chunk "read" flag;
//   * before writing, it waits until every earlier chunk whose source rows
//     reach into its destination rows has published its flag.
// Sources of a destination row j lie at j + shift >= j, so a chunk's writes
// can only clobber sources of earlier chunks (or its own, which it already
// holds).  Blocks wait only on chunks with earlier tickets, which are
// resident or finished, so the waits always end; each wait is still bounded
// and reports kErrWait instead of spinning forever.
#include "kvm_internal.cuh"

namespace kvm {
namespace {

constexpr int kWaitLimit = 1 << 22;   // ~0.3-1 s with the back-off below

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Old (source) index of new index j >= first, for one character.
__device__ __forceinline__ int src_index(const int32_t* seg_start, const int32_t* seg_shift,
                                         int n_seg, int j) {
    int lo = 0, hi = n_seg - 1;            // last k with seg_start[k] <= j
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (seg_start[mid] <= j) lo = mid; else hi = mid - 1;
    }
    return j + seg_shift[lo];
}

__global__ void __launch_bounds__(kCompactThreads)
kv_compact_kernel(const __grid_constant__ CompactParams p) {
    const int tid = threadIdx.x;
    // character of this block: last b with blk_off <= blockIdx.x
    int lo = 0, hi = p.n_chars - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (p.ch[mid].blk_off <= (int)blockIdx.x) lo = mid; else hi = mid - 1;
    }
    const int b = lo;
    const CompactChar& c = p.ch[b];
    const int local = blockIdx.x - c.blk_off;
    const bool is_pos = local >= p.n_kv_slabs * c.chunks_kv;
    const int slab = is_pos ? p.n_kv_slabs : local / c.chunks_kv;
    const int n_chunks = is_pos ? c.chunks_pos : c.chunks_kv;
    const int rows = is_pos ? p.rows_pos : p.rows_kv;
    const int32_t* seg_start = p.seg_start + c.seg_off;
    const int32_t* seg_shift = p.seg_shift + c.seg_off;

    __shared__ int s_chunk;
    __shared__ int s_abort;
    if (tid == 0) {
        int32_t* counter = p.tickets + b * (p.n_kv_slabs + 1) + slab;
        int t = atomicAdd(counter, 1);
        if (t == n_chunks - 1) atomicExch(counter, 0);   // every ticket of this launch is taken
        s_chunk = t;
        s_abort = 0;
        if (t >= n_chunks) { atomicOr(p.err, kErrBounds); s_abort = 1; }
    }
    __syncthreads();
    if (s_abort) return;
    const int chunk = s_chunk;
    const int d0 = c.first + chunk * rows;
    const int d1 = min(d0 + rows, c.L_new);
    const int flag_base = c.flag_off + slab * c.chunks_kv;   // pos slab follows the KV slabs

    uint4 vbuf[kCompactVecPerThread];
    int32_t ibuf[kCompactVecPerThread];
    uint4* base = nullptr;
    if (!is_pos) {
        const int half = p.n_kv_slabs / 2;
        uint4* arr = slab < half ? p.K : p.V;
        const int s_in = slab < half ? slab : slab - half;
        base = arr + ((int64_t)s_in * p.slab_rows + c.cap_off) * p.vec_per_row;
        const int n_vec = (d1 - d0) * p.vec_per_row;
#pragma unroll
        for (int k = 0; k < kCompactVecPerThread; ++k) {
            const int v = tid + k * kCompactThreads;
            if (v < n_vec) {
                const int row = d0 + v / p.vec_per_row;
                const int src = src_index(seg_start, seg_shift, c.n_seg, row);
                vbuf[k] = __ldcg(base + (int64_t)src * p.vec_per_row + v % p.vec_per_row);
            }
        }
    } else {
#pragma unroll
        for (int k = 0; k < kCompactVecPerThread; ++k) {
            const int row = d0 + tid + k * kCompactThreads;
            if (row < d1) {
                const int src = src_index(seg_start, seg_shift, c.n_seg, row);
                ibuf[k] = __ldcg(p.pos + c.cap_off + src);
            }
        }
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) {
        st_release(p.flags + flag_base + chunk, p.epoch);
        // wait for earlier chunks whose sources reach into [d0, d1)
        for (int e = chunk - 1; e >= 0; --e) {
            const int last_dst = min(c.first + (e + 1) * rows, c.L_new) - 1;
            if (src_index(seg_start, seg_shift, c.n_seg, last_dst) < d0) break;
            int it = 0;
            while (ld_acquire(p.flags + flag_base + e) != p.epoch) {
                if (++it > kWaitLimit) { atomicOr(p.err, kErrWait); s_abort = 1; break; }
                __nanosleep(64);
            }
            if (s_abort) break;
        }
    }
    __syncthreads();
    if (s_abort) return;

    if (!is_pos) {
        const int n_vec = (d1 - d0) * p.vec_per_row;
#pragma unroll
        for (int k = 0; k < kCompactVecPerThread; ++k) {
            const int v = tid + k * kCompactThreads;
            if (v < n_vec) __stcg(base + (int64_t)d0 * p.vec_per_row + v, vbuf[k]);
        }
    } else {
#pragma unroll
        for (int k = 0; k < kCompactVecPerThread; ++k) {
            const int row = d0 + tid + k * kCompactThreads;
            if (row < d1) __stcg(p.pos + c.cap_off + row, ibuf[k]);
        }
    }
}

__global__ void gather_map_kernel(const __grid_constant__ GatherParams p) {
    for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < p.total; idx += gridDim.x * blockDim.x) {
        int lo = 0, hi = p.n_chars - 1;
        while (lo < hi) {
            int mid = (lo + hi + 1) >> 1;
            if (p.out_off[mid] <= idx) lo = mid; else hi = mid - 1;
        }
        const int j = idx - p.out_off[lo];
        int src = j;
        if (p.n_seg[lo] > 0 && j >= p.first[lo])
            src = src_index(p.seg_start + p.seg_off[lo], p.seg_shift + p.seg_off[lo], p.n_seg[lo], j);
        p.out[idx] = src;
    }
}

}  // namespace

void launch_kv_compact(const CompactParams& p, cudaStream_t s) {
    if (p.total_blocks <= 0) return;
    kv_compact_kernel<<<p.total_blocks, kCompactThreads, 0, s>>>(p);
}

void launch_gather_map(const GatherParams& p, cudaStream_t s) {
    if (p.total <= 0) return;
    int blocks = (p.total + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    gather_map_kernel<<<blocks, 256, 0, s>>>(p);
}

}  // namespace kvm
