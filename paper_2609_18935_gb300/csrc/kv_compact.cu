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
#include <cstdio>
#include <cstring>

#include "kvm_internal.cuh"

namespace kvm {
namespace {

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
    grid_dependency_wait();
    grid_dependents_launch();
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
    if (tid == 0) st_release(p.flags + (int64_t)(flag_base + chunk) * p.flag_stride, p.epoch);
    if (tid < 32) {
        // earlier chunks whose sources reach into [d0, d1) are e_min .. chunk - 1
        // (their last sources are ordered); the lanes of warp 0 wait on their
        // flags together, one flag each, so the waits cost one round trip
        int e_min = chunk;
        for (int e = chunk - 1; e >= 0; --e) {
            const int last_dst = min(c.first + (e + 1) * rows, c.L_new) - 1;
            if (src_index(seg_start, seg_shift, c.n_seg, last_dst) < d0) break;
            e_min = e;
        }
        bool fail = false;
        for (int e = e_min + tid; e < chunk && !fail; e += 32) {
            int it = 0;
            while (ld_acquire(p.flags + (int64_t)(flag_base + e) * p.flag_stride) != p.epoch) {
                if (++it > p.wait_limit) { fail = true; break; }
                __nanosleep(64);
            }
        }
        if (p.never_set && tid == 0) {
            int it = 0;
            while (ld_acquire(p.never_set) != p.epoch) {
                if (++it > p.wait_limit) { fail = true; break; }
                __nanosleep(64);
            }
        }
        if (__any_sync(0xffffffffu, fail) && tid == 0) {
            atomicOr(p.err, kErrWait);
            s_abort = 1;
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
    grid_dependency_wait();
    grid_dependents_launch();
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
    launch_pdl(kv_compact_kernel, dim3(p.total_blocks), dim3(kCompactThreads), 0, s, p);
}

void launch_gather_map(const GatherParams& p, cudaStream_t s) {
    if (p.total <= 0) return;
    int blocks = (p.total + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    launch_pdl(gather_map_kernel, dim3(blocks), dim3(256), 0, s, p);
}

}  // namespace kvm

// ============================================================================
// Allocation-free compaction of caller-owned KV slabs.
//
// For callers that cannot call cudaMalloc: for example a game engine that
// owns all device memory through its own fixed arena and forbids other
// allocations during a session, or a frame loop in which an allocation (which
// may synchronize the device) would stall the frame.  Such callers cannot
// create a kvm context (kvm_create allocates), so this entry point compacts
// KV buffers they own, and keeps the few words of bookkeeping the kernel
// needs (per-slab tickets, per-chunk read flags, an error word) in the
// fixed-size device array below instead of allocated workspace.  That array
// lives in every GPU that loads the library until the process exits.
// ============================================================================
#include "../../include/kvm.h"

namespace {
constexpr int kNoAllocMaxSlabs = 512;                       // K slabs (layers x KV heads), V slabs as many
constexpr int kNoAllocTickets = 2 * kNoAllocMaxSlabs + 1;   // + the position slab
constexpr int kNoAllocMaxFlags = 65536;                     // read flags (one per moved chunk per slab)
constexpr int kNoAllocWords = 64 + kNoAllocTickets + kNoAllocMaxFlags;   // word 0: device error word
constexpr int kMaxDevices = 64;
}  // namespace

static __device__ __align__(256) uint32_t kvm_noalloc_scratch[kNoAllocWords];

namespace {
// Device address of kvm_noalloc_scratch per device, found once per device
// (the name is a host-side stand-in; only cudaGetSymbolAddress gives the
// address a kernel can use).
uint32_t* g_noalloc_addr[kMaxDevices] = {};
}  // namespace

extern "C" kvm_status kvm_kv_compact_noalloc(void* K, void* V, int32_t* positions, int32_t n_slabs,
                                             int64_t slab_rows, int32_t head_dim, int32_t live,
                                             int32_t n_spans, const int32_t* span_begin,
                                             const int32_t* span_end, int32_t* new_live_out, void* stream) {
    using namespace kvm;
    if (!K || !V) return report_error(KVM_E_INVAL, "kv_compact_noalloc: K or V is NULL");
    if (n_slabs <= 0 || n_slabs > kNoAllocMaxSlabs)
        return report_error(KVM_E_CAPACITY, "kv_compact_noalloc: n_slabs must be in [1, 512]");
    if (head_dim != 64 && head_dim != 128 && head_dim != 256)
        return report_error(KVM_E_UNSUPPORTED, "kv_compact_noalloc: head_dim must be 64, 128 or 256");
    if (live < 0 || slab_rows < live || slab_rows > INT32_MAX)
        return report_error(KVM_E_INVAL, "kv_compact_noalloc: need 0 <= live <= slab_rows <= 2^31-1");
    if (n_spans < 0 || n_spans > kMaxSpans)
        return report_error(KVM_E_CAPACITY, "kv_compact_noalloc: n_spans must be in [0, 1024]");
    if (n_spans > 0 && (!span_begin || !span_end))
        return report_error(KVM_E_INVAL, "kv_compact_noalloc: span arrays are NULL");
    if (!new_live_out) return report_error(KVM_E_INVAL, "kv_compact_noalloc: new_live_out is NULL");

    thread_local static CompactParams p;
    std::memset(&p, 0, sizeof p);
    int removed = 0, prev_end = 0;
    for (int k = 0; k < n_spans; ++k) {
        const int lo = span_begin[k], hi = span_end[k];
        if (!(0 <= lo && lo < hi && hi <= live))
            return report_error(KVM_E_SPAN, "kv_compact_noalloc: span empty or outside the live rows");
        if (k > 0 && lo < prev_end)
            return report_error(KVM_E_SPAN, "kv_compact_noalloc: spans must be sorted and disjoint");
        prev_end = hi;
        removed += hi - lo;
        p.seg_start[k] = hi - removed;
        p.seg_shift[k] = removed;
    }
    const int L_new = live - removed;
    const int vec_per_row = head_dim * 2 / 16;
    const int rows_kv = kCompactVecPerChunk / vec_per_row;
    const int rows_pos = kCompactVecPerChunk;
    const int moved = n_spans > 0 ? L_new - span_begin[0] : 0;
    const int chunks_kv = (moved + rows_kv - 1) / rows_kv;
    const int chunks_pos = positions ? (moved + rows_pos - 1) / rows_pos : 0;
    const int64_t n_flags = (int64_t)2 * n_slabs * chunks_kv + chunks_pos;
    if (n_flags > kNoAllocMaxFlags)
        return report_error(KVM_E_CAPACITY,
                            "kv_compact_noalloc: 2 * n_slabs * ceil(moved / rows_per_chunk) + position chunks "
                            "exceeds the 65536 read flags of the static scratch");

    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return report_error(KVM_E_CUDA, "kv_compact_noalloc: no usable current device");
    if (!g_noalloc_addr[dev]) {
        void* addr = nullptr;
        e = cudaGetSymbolAddress(&addr, kvm_noalloc_scratch);
        if (e != cudaSuccess || !addr)
            return report_error(KVM_E_CUDA, "kv_compact_noalloc: cudaGetSymbolAddress of the scratch failed");
        g_noalloc_addr[dev] = static_cast<uint32_t*>(addr);
    }
    uint32_t* scratch = g_noalloc_addr[dev];
    *new_live_out = L_new;
    if (moved <= 0) return KVM_OK;

    cudaStream_t s = (cudaStream_t)stream;
    // tickets and the flags this call uses start at zero (the array keeps the
    // previous call's contents); epoch 1 then marks "chunk read"
    uint32_t* tickets = scratch + 64;
    uint32_t* flags = tickets + kNoAllocTickets;
    e = cudaMemsetAsync(tickets, 0, sizeof(uint32_t) * (2 * n_slabs + 1), s);
    if (e == cudaSuccess) e = cudaMemsetAsync(flags, 0, sizeof(uint32_t) * (size_t)n_flags, s);
    if (e != cudaSuccess) return report_error(KVM_E_CUDA, "kv_compact_noalloc: clearing the scratch failed");

    p.n_chars = 1;
    p.n_kv_slabs = 2 * n_slabs;
    p.vec_per_row = vec_per_row;
    p.rows_kv = rows_kv;
    p.rows_pos = rows_pos;
    p.epoch = 1;
    p.slab_rows = slab_rows;
    p.K = static_cast<uint4*>(K);
    p.V = static_cast<uint4*>(V);
    p.pos = positions;
    p.tickets = reinterpret_cast<int32_t*>(tickets);
    p.flags = flags;
    p.flag_stride = 1;
    p.err = reinterpret_cast<int32_t*>(scratch);
    p.wait_limit = kCompactWaitLimit;
    CompactChar& c = p.ch[0];
    c.L_new = L_new;
    c.first = span_begin[0];
    c.seg_off = 0;
    c.n_seg = n_spans;
    c.cap_off = 0;
    c.chunks_kv = chunks_kv;
    c.chunks_pos = chunks_pos;
    c.blk_off = 0;
    c.flag_off = 0;
    p.total_blocks = p.n_kv_slabs * chunks_kv + chunks_pos;
    launch_kv_compact(p, s);
    e = cudaGetLastError();
    if (e != cudaSuccess) return report_error(KVM_E_CUDA, "kv_compact_noalloc: kernel launch failed");
    return KVM_OK;
}

extern "C" kvm_status kvm_kv_compact_noalloc_check(void* stream) {
    using namespace kvm;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return report_error(KVM_E_CUDA, "kv_compact_noalloc_check: no usable current device");
    // no call on this device yet: nothing can have failed
    if (!g_noalloc_addr[dev]) return KVM_OK;
    e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return report_error(KVM_E_CUDA, "kv_compact_noalloc_check: stream synchronize failed");
    uint32_t word = 0;
    e = cudaMemcpy(&word, g_noalloc_addr[dev], sizeof word, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return report_error(KVM_E_CUDA, "kv_compact_noalloc_check: reading the error word failed");
    if (!word) return KVM_OK;
    e = cudaMemset(g_noalloc_addr[dev], 0, sizeof word);
    if (e != cudaSuccess) return report_error(KVM_E_CUDA, "kv_compact_noalloc_check: clearing the error word failed");
    char msg[160];
    snprintf(msg, sizeof msg, "kv_compact_noalloc: device error word 0x%x (%s%s); the rows of the failed call are undefined",
             word, (word & kErrBounds) ? "bounds " : "", (word & kErrWait) ? "wait-timeout" : "");
    return report_error(KVM_E_DEVICE, msg);
}
