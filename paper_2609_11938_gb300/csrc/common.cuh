// common.cuh -- context, scratch arena, launch accounting and device helpers
// shared by the kernels of libopattr.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <string>
#include <vector>

#include "opattr.h"

namespace opattr {

// ------------------------------------------------------------------ status block
// One small struct in device memory per context, reset at the start of each
// call and read back at its checkpoints.  Kernels never trap: they record
// problems here and return.
enum ErrBit : unsigned {
    ERR_INVALID = 1u,     // bad id, value or size found on the device
    ERR_NOT_NESTED = 2u,  // ranges are not laminar
    ERR_DEPTH = 4u,       // depth > 31
    ERR_TIMEOUT = 8u,     // a bounded wait gave up
    ERR_COUNT = 16u,      // count mismatch in error mode
};
enum FlagBit : unsigned {
    F_K_UNSORTED = 1u,    // kernels are not in (start, stream) order
    F_R_UNSORTED = 2u,    // ranges are not in start order
    F_LEVEL_FIXUP = 4u,   // equal starts in a level are not in end order
    F_NAMES_DIFFER = 8u,  // ncu names differ from replayed names in time order
    F_OP_DUP = 16u,       // two operator ranges share an op id
    F_AGG_MISS = 32u,     // the owned-range aggregation missed kernels
    F_IDX_NOT_ID = 64u,   // some kernel's ncu row index is neither its own index nor -1
};
enum CountSlot {
    C_NAMES_MISMATCH = 0,
    C_COUNT_UNMATCHED,
    C_DIRECT,
    C_BROADCAST,
    C_DEDUP_MISMATCH,
    C_REPLAYED,
    C_TOTAL_NS,
    C_ATTR_NS,
    C_ATTR_K,
    C_MATCHED_K,
    C_AGG_SEEN,
    C_UNMATCHED,
    C_TIER_HIGH,
    C_TIER_NVTX,
    C_TIER_INDUCTOR,
    C_FUSED,
    C_CORR_USED,
    C_NSLOTS = 24
};
enum MinMaxSlot { MM_KSTART_MIN = 0, MM_KSTART_MAX, MM_RSTART_MIN, MM_REND_MAX, MM_NSLOTS = 8 };

struct DevStatus {
    unsigned int err;
    unsigned int flags;
    unsigned long long cnt[C_NSLOTS];
    long long mm[MM_NSLOTS];
};

// ------------------------------------------------------------------ context
struct TimingSlot {
    const char *name;
    double total_ms;
    int64_t launches;
};

constexpr int N_LEVELS = 256 * 32;   // (stream, depth) levels of the enclosure
constexpr size_t STAGE_BYTES = 32768;  // pinned staging of host-built tables (one copy per call)

struct Ctx {
    int device = 0;
    cudaStream_t stream = nullptr;
    // a second stream for independent chains of one call (the enclosure's
    // level lists beside its stream partition), with the events that fork
    // from and join back into `stream`; created on first use
    cudaStream_t side = nullptr;
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr, ev_join2 = nullptr;
    opattr_config cfg{};
    bool broken = false;
    // scratch arena (bump allocation, reset per call)
    char *arena = nullptr;
    size_t arena_cap = 0, arena_used = 0;
    bool arena_fixed = false;        // the arena is caller-provided memory: never grow or free it
    // status block
    DevStatus *d_status = nullptr;
    DevStatus *h_status = nullptr;   // pinned mirror
    DevStatus *h_init = nullptr;     // pinned reset template
    uint32_t *h_levels = nullptr;    // pinned host copy of the enclosure's level offsets [N_LEVELS + 1] and
                                     // kernels per stream [256];
                                     // the aggregation reuses it for a few values read mid-call
    unsigned char *h_stage = nullptr; // pinned staging for small host-built tables [STAGE_BYTES]
    bool host_mapped = false;        // the four pinned buffers above are addressable from the device as they are
    // kernel time order as the last enclosure found it (-1 unknown, 0 / 1),
    // and whether the matching may take it instead of checking again (join)
    int enclose_k_sorted = -1;
    bool order_from_enclose = false;
    // within a join: the enclosure's kernel time order (unsorted kernels), kept
    // for the matching at the start of the arena (arena_keep bytes survive the
    // per-call resets and any growth of the arena)
    bool in_join = false;
    uint32_t *join_korder = nullptr;
    size_t arena_keep = 0;
    // launch accounting
    // within a join: the matching's identity pairing (rows equal to the
    // kernels in time order), launched beside the enclosure when spec_k > 0;
    // spec_ran: it ran in the enclosure's last attempt, its verdict in the
    // status the enclosure read last
    const uint32_t *spec_kname = nullptr, *spec_nname = nullptr;
    int32_t *spec_idx = nullptr;
    uint8_t *spec_kind = nullptr;
    int64_t spec_k = 0;
    bool spec_ran = false;
    // within a join whose matching can be skipped: the enclosure's last status
    // read is left to the aggregation's (defer_status), and the enclosure's
    // verdict is pending until then (enclose_pending; the aggregation keeps
    // the status block instead of resetting it)
    bool defer_status = false, enclose_pending = false;
    // within a join: the matching was the identity pairing (row k for kernel
    // k), so the aggregation need not read the row indices
    bool rows_identity = false;
    int64_t launches = 0;
    bool timing = false;
    std::string timing_only;         // with timing on: bracket only this kernel (empty = all)
    std::vector<TimingSlot> slots;
    std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> pending;
    std::vector<cudaEvent_t> event_pool;
    cudaError_t last_error = cudaSuccess;
};

// ------------------------------------------------------------------ scratch
struct Arena {
    Ctx &c;
    explicit Arena(Ctx &ctx) : c(ctx) { c.arena_used = c.arena_keep; }
    template <typename T>
    T *take(int64_t count) {
        size_t bytes = (size_t)(count > 0 ? count : 1) * sizeof(T);
        size_t at = (c.arena_used + 255) & ~(size_t)255;
        if (at + bytes > c.arena_cap) return nullptr;
        c.arena_used = at + bytes;
        return reinterpret_cast<T *>(c.arena + at);
    }
};
// Upper bound of an arena request made of several arrays (alignment slack included).
struct Need {
    size_t bytes = 0;
    template <typename T>
    Need &add(int64_t count) {
        bytes += (((size_t)(count > 0 ? count : 1) * sizeof(T)) + 255) & ~(size_t)255;
        return *this;
    }
};

opattr_status ensure_arena(Ctx &c, size_t bytes);
opattr_status ensure_side(Ctx &c);       // the side stream and its events
// Algorithm 1's identity pairing on c.stream (match.cu): kernel j's row is
// row j, F_NAMES_DIFFER set where the names disagree
void launch_identity_match(Ctx &c, const uint32_t *kname, const uint32_t *nname, int64_t K, int32_t *out_idx,
                           uint8_t *out_kind);

// Launches and async copies within the scope go to stream s (c.stream is
// swapped and restored).
struct OnStream {
    Ctx &c;
    cudaStream_t prev;
    OnStream(Ctx &ctx, cudaStream_t s) : c(ctx), prev(ctx.stream) { c.stream = s; }
    ~OnStream() { c.stream = prev; }
    OnStream(const OnStream &) = delete;
    OnStream &operator=(const OnStream &) = delete;
};
// `to` waits for the work issued to `from` so far (through event e).
inline void stream_after(cudaStream_t to, cudaStream_t from, cudaEvent_t e) {
    cudaEventRecord(e, from);
    cudaStreamWaitEvent(to, e, 0);
}
// A small transfer between the context's pinned host buffers and device
// memory, on c.stream.  When those buffers are mapped into the device's
// address space (opattr_create checks), a small kernel moves the bytes through
// the mapping instead of a copy engine, so a call's status reads and table
// uploads never queue behind bulk copies that the caller has on the engines;
// otherwise (host mirrors in plain host memory) cudaMemcpyAsync.
opattr_status copy_small(Ctx &c, void *dst, const void *src, size_t bytes, cudaMemcpyKind kind);
struct SmallCopy {
    void *dst;
    const void *src;
    size_t bytes;
};
// Several such transfers of one direction, four to a launch.
opattr_status copy_small_n(Ctx &c, int count, const SmallCopy *cp, cudaMemcpyKind kind);
opattr_status reset_status(Ctx &c);
// The status block back to the host (with up to three more device->host
// transfers in the same launch), then a stream synchronize.
opattr_status read_status(Ctx &c, int n_extra = 0, const SmallCopy *extra = nullptr);
opattr_status cuda_status(Ctx &c, cudaError_t e);
int timing_slot(Ctx &c, const char *name);
void timing_begin(Ctx &c, int slot, cudaEvent_t *e0, cudaEvent_t *e1);
void timing_end(Ctx &c, int slot, cudaEvent_t e0, cudaEvent_t e1);
void timing_collect(Ctx &c);             // after a stream synchronize

// Launch a kernel on the context stream, counting it and (optionally) timing
// it.  Kernels go out as programmatic dependent launches: the next kernel of
// the stream is set up and its blocks scheduled while this one's last blocks
// finish, instead of after its completion; every kernel of the library calls
// pdl_wait() before its first memory access, which holds it until the
// kernel before it has completed and its writes are visible.
template <typename... KArgs, typename... Args>
inline void launch(Ctx &c, const char *name, void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                   Args... args) {
    if (grid.x == 0 || grid.y == 0 || grid.z == 0) return;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    int slot = -1;
    const bool timed = c.timing && (c.timing_only.empty() || c.timing_only == name);
    if (timed) {
        slot = timing_slot(c, name);
        timing_begin(c, slot, &e0, &e1);
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = c.stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaLaunchKernelEx(&cfg, kern, args...);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess && c.last_error == cudaSuccess) c.last_error = e;
    c.launches++;
    if (timed) timing_end(c, slot, e0, e1);
}

inline unsigned grid_for(int64_t n, int per_block, unsigned cap = 1u << 30) {
    int64_t g = (n + per_block - 1) / per_block;
    if (g < 1) g = 1;
    return (unsigned)(g > (int64_t)cap ? cap : g);
}

// ------------------------------------------------------------------ device helpers
// The first statement of every kernel: waits, under a programmatic dependent
// launch, until the kernel before it in the stream has completed and its
// memory is visible (returns at once otherwise).  No kernel signals early
// completion, so a kernel's blocks never hold resources that the blocks of
// the kernel before it still need.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ unsigned lane_id() { return threadIdx.x & 31u; }
__device__ __forceinline__ unsigned lanemask_lt() {
    unsigned m;
    asm volatile("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// Lanes of the warp whose 8-bit digit equals this lane's, among the lanes
// with `valid` set: one ballot per digit bit (the rank-by-digit step of a
// stable multi-split).
__device__ __forceinline__ unsigned warp_peers8(unsigned d, bool valid) {
    unsigned m = __ballot_sync(0xffffffffu, valid);
#pragma unroll
    for (int b = 0; b < 8; ++b) {
        const bool bit = (d >> b) & 1u;
        const unsigned x = __ballot_sync(0xffffffffu, bit);
        m &= bit ? x : ~x;
    }
    return m;
}

__device__ __forceinline__ void set_err(DevStatus *s, unsigned bit) { atomicOr(&s->err, bit); }
__device__ __forceinline__ void set_flag(DevStatus *s, unsigned bit) { atomicOr(&s->flags, bit); }

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
template <typename T>
__device__ __forceinline__ T warp_inclusive_scan(T v) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        T u = __shfl_up_sync(0xffffffffu, v, o);
        if ((int)lane_id() >= o) v += u;
    }
    return v;
}

// Exclusive scan over a block (blockDim.x a multiple of 32, <= 1024).
// `warp_buf` holds 33 entries of shared memory.  Returns the exclusive prefix;
// *total receives the block sum.
template <typename T>
__device__ __forceinline__ T block_exclusive_scan(T v, T *warp_buf, T *total) {
    const unsigned w = threadIdx.x >> 5, nw = blockDim.x >> 5;
    T inc = warp_inclusive_scan(v);
    if (lane_id() == 31) warp_buf[w] = inc;
    __syncthreads();
    if (w == 0) {
        T x = lane_id() < nw ? warp_buf[lane_id()] : T(0);
        T xs = warp_inclusive_scan(x);
        if (lane_id() < nw) warp_buf[lane_id()] = xs - x;
        if (lane_id() == nw - 1) warp_buf[32] = xs;
    }
    __syncthreads();
    T r = warp_buf[w] + inc - v;
    if (total) *total = warp_buf[32];
    __syncthreads();
    return r;
}

template <typename T>
__device__ __forceinline__ T block_sum(T v, T *warp_buf) {
    T total;
    block_exclusive_scan(v, warp_buf, &total);
    return total;
}

// Sum v over the block and add the total to *dst with one atomic.  Every
// thread of the block must call it (it synchronises the block).
__device__ __forceinline__ void block_add_u64(unsigned long long v, unsigned long long *dst,
                                              unsigned long long *warp_buf) {
    unsigned long long t = block_sum<unsigned long long>(v, warp_buf);
    if (threadIdx.x == 0 && t) atomicAdd(dst, t);
}

// Stable grouping of a block's entries by key.  The block's warps own
// consecutive runs of PER_WARP entries; entry i has key key_of(i) < nkeys or
// GROUP_NONE.  On return soff[0..nkeys] hold the group offsets and klist the
// entry indices grouped by key, in index order within a group.  wcnt is a
// [warps][wstride] scratch of 16-bit counters (wstride >= nkeys).  Warps rank
// their entries 32 at a time with __match_any_sync peer groups.  Every thread
// of the block must call it; it ends with a barrier.
constexpr unsigned GROUP_NONE = 0xFFFFu;
template <int THREADS, int PER_WARP, typename KeyFn>
__device__ __forceinline__ void block_group_by_key(int nkeys, KeyFn key_of, uint16_t *wcnt, int wstride,
                                                   uint16_t *soff, uint16_t *klist, uint32_t *wbuf) {
    constexpr int WARPS = THREADS / 32;
    const unsigned w = threadIdx.x >> 5, lane = lane_id(), lt = lanemask_lt();
    for (int q = 0; q < WARPS; ++q)
        for (int k = threadIdx.x; k < nkeys; k += THREADS) wcnt[q * wstride + k] = 0;
    __syncthreads();
    uint16_t rank[PER_WARP / 32];
    uint16_t key[PER_WARP / 32];
#pragma unroll
    for (int it = 0; it < PER_WARP / 32; ++it) {
        const int i = w * PER_WARP + it * 32 + lane;
        const unsigned k = key_of(i);
        const unsigned peers = __match_any_sync(0xffffffffu, k);
        const unsigned before = k != GROUP_NONE ? wcnt[w * wstride + k] : 0u;
        __syncwarp();
        if (k != GROUP_NONE && (peers & lt) == 0) wcnt[w * wstride + k] = (uint16_t)(before + __popc(peers));
        __syncwarp();
        rank[it] = (uint16_t)(before + __popc(peers & lt));
        key[it] = (uint16_t)k;
    }
    __syncthreads();
    unsigned carry = 0;
    for (int b = 0; b < nkeys; b += THREADS) {
        const int k = b + threadIdx.x;
        unsigned tot = 0;
        if (k < nkeys) {
#pragma unroll
            for (int q = 0; q < WARPS; ++q) {
                unsigned x = wcnt[q * wstride + k];
                wcnt[q * wstride + k] = (uint16_t)tot;
                tot += x;
            }
        }
        unsigned all;
        const unsigned ex = block_exclusive_scan<unsigned>(tot, wbuf, &all);
        if (k < nkeys) soff[k] = (uint16_t)(carry + ex);
        carry += all;
    }
    if (threadIdx.x == 0) soff[nkeys] = (uint16_t)carry;
    __syncthreads();
#pragma unroll
    for (int it = 0; it < PER_WARP / 32; ++it) {
        const unsigned k = key[it];
        if (k != GROUP_NONE) klist[soff[k] + wcnt[w * wstride + k] + rank[it]] = (uint16_t)(w * PER_WARP + it * 32 + lane);
    }
    __syncthreads();
}

// Blocks for grid-stride reductions: enough to fill the GPU, few enough that
// one atomic per block stays cheap.
constexpr unsigned REDUCE_GRID = 2048;

}  // namespace opattr
