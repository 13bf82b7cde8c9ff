// enclose.cu -- Algorithm 2 (NVTX enclosure attribution, Sec. 3.5) on the GPU.
//
// Data layout.  Ranges are regrouped into per-(stream, depth) level lists,
// each in (start, end, index) order: lvl_start / lvl_end (i64) and lvl_info
// (u32: range index in the low 30 bits, kind in the top 2: 0 operator,
// 1 non-op, 2 structural).  lvl_off[level] gives the list bounds, level =
// stream * 32 + depth.  Within a level ranges are disjoint or touching, so
// "the last range with start <= T" is the only one that can contain T.
//
// Kernels are answered stream by stream, in tiles of consecutive kernels of
// one stream (the per-stream tiles section below).  A window table bounds,
// per tile and depth, the ranges the tile can hit; the enclosure kernel
// stages those windows in shared memory as 32-bit times relative to the
// tile's first kernel and sweeps the tile's kernels in time order, walking
// depths outward-in (0, 1, ...) until a depth has no containing range.  The
// walk state needs no stack: a structural range resets the collection
// (everything above it is beyond the cut); an operator becomes the innermost
// answer and counts; a non-op range is passed over.
#include <algorithm>

#include "sort.cuh"
#include "util.cuh"

namespace opattr {

constexpr int LEVELS = N_LEVELS;
constexpr uint32_t KIND_OP = 0, KIND_NONOP = 1, KIND_STRUCT = 2;

__device__ __forceinline__ uint32_t kind_of(uint32_t op) {
    return op == OPATTR_OP_STRUCTURAL ? KIND_STRUCT : (op == OPATTR_OP_NONOP ? KIND_NONOP : KIND_OP);
}

// ------------------------------------------------------------------ range checks
// end >= start, depth <= 31, start order of the array, min start / max end,
// and a histogram of level keys (per block in shared memory, flushed with
// one global atomic per non-empty bin).
constexpr int RCHK_THREADS = 256;
constexpr int RCHK_ITEMS = 16;
__global__ void __launch_bounds__(RCHK_THREADS) k_check_ranges(const uint8_t *__restrict__ stream,
                                                               const int64_t *__restrict__ start,
                                                               const int64_t *__restrict__ end,
                                                               const uint8_t *__restrict__ depth, int64_t n,
                                                               uint32_t *__restrict__ level_hist, DevStatus *st) {
    pdl_wait();
    __shared__ uint32_t h[LEVELS];
    __shared__ int flags;
    __shared__ long long smin, smax;
    for (int i = threadIdx.x; i < LEVELS; i += RCHK_THREADS) h[i] = 0;
    if (threadIdx.x == 0) { flags = 0; smin = LLONG_MAX; smax = LLONG_MIN; }
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RCHK_THREADS * RCHK_ITEMS;
    long long mn = LLONG_MAX, mx = LLONG_MIN;
    int f = 0;
    constexpr int B = 4;                    // items per batch, loads issued together
    for (int it0 = 0; it0 < RCHK_ITEMS; it0 += B) {
        long long sv[B], ev[B], nv[B];
        unsigned dv[B], stv[B];
#pragma unroll
        for (int u = 0; u < B; ++u) {
            const int64_t i = base + (it0 + u) * RCHK_THREADS + threadIdx.x;
            const bool in = i < n;
            sv[u] = in ? start[i] : 0;
            ev[u] = in ? end[i] : 0;
            nv[u] = i + 1 < n ? start[i + 1] : LLONG_MAX;
            dv[u] = in ? depth[i] : 0u;
            stv[u] = in ? stream[i] : 0u;
        }
#pragma unroll
        for (int u = 0; u < B; ++u) {
            const int64_t i = base + (it0 + u) * RCHK_THREADS + threadIdx.x;
            if (i >= n) continue;
            if (ev[u] < sv[u]) f |= 1;
            if (dv[u] >= OPATTR_MAX_DEPTH) f |= 2;
            if (nv[u] < sv[u]) f |= 4;
            mn = sv[u] < mn ? sv[u] : mn;
            mx = ev[u] > mx ? ev[u] : mx;
            if (dv[u] < OPATTR_MAX_DEPTH) atomicAdd(&h[stv[u] * 32 + dv[u]], 1u);
        }
    }
    if (f) atomicOr(&flags, f);
    atomicMin(&smin, mn);
    atomicMax(&smax, mx);
    __syncthreads();
    for (int i = threadIdx.x; i < LEVELS; i += RCHK_THREADS)
        if (h[i]) atomicAdd(&level_hist[i], h[i]);
    if (threadIdx.x == 0) {
        if (flags & 1) set_err(st, ERR_INVALID);
        if (flags & 2) set_err(st, ERR_DEPTH);
        if (flags & 4) set_flag(st, F_R_UNSORTED);
        atomicMin(&st->mm[MM_RSTART_MIN], smin);
        atomicMax(&st->mm[MM_REND_MAX], smax);
    }
}

// ------------------------------------------------------------------ level lists
__global__ void k_level_keys(const uint8_t *__restrict__ stream, const uint8_t *__restrict__ depth,
                             const uint32_t *__restrict__ perm, int64_t n, uint32_t *__restrict__ keys) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = perm ? perm[i] : i;
        keys[i] = (uint32_t)stream[r] * 32u + depth[r];
    }
}
// The level lists' order key of range i: its start, then 0 for a
// zero-length range and 1 for a longer one.  Within a level of laminar
// ranges two ranges share a start only if all but the last of them have
// zero length, so a stable sort on this key puts every level in (start,
// end, index) order -- the order of Algorithm 2's one representative per
// depth -- in one sort; two longer ranges sharing a start in one level are
// out of that order only when they overlap, which the validation reports.
__global__ void k_range_start_key(const int64_t *__restrict__ start, const int64_t *__restrict__ end, int64_t n,
                                  long long tmin, uint64_t *__restrict__ keys) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        keys[i] = ((uint64_t)(start[i] - tmin) << 1) | (end[i] > start[i] ? 1u : 0u);
}
__global__ void k_level_gather(const int64_t *__restrict__ start, const int64_t *__restrict__ end,
                               const uint32_t *__restrict__ op, const uint32_t *__restrict__ perm, int64_t n,
                               int64_t *__restrict__ ls, int64_t *__restrict__ le, uint32_t *__restrict__ li) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t r = perm[i];
        ls[i] = start[r];
        le[i] = end[r];
        li[i] = r | (kind_of(op[r]) << 30);
    }
}

// The same partition in one counting pass when at most 256 levels are
// present: range i's digit is its compact level id (levels numbered in
// (stream, depth) order, so a stable partition by compact id is the stable
// sort by level key), and k_level_place writes each range's level-list
// entry in place of the key sort and the gather.
struct LevelDigit {
    const uint8_t *stream, *depth;
    const uint8_t *cmap;        // [LEVELS] compact id of each present level
    const uint32_t *perm;       // NULL = array order
    __device__ __forceinline__ unsigned operator()(int64_t i) const {
        const uint32_t r = perm ? perm[i] : (uint32_t)i;
        return cmap[stream[r] * 32u + depth[r]];
    }
};
// The placing pass: the digit-rank of the tile's ranges gives each its
// place in the tile sorted by compact level; the range's tile index is
// staged there in shared memory, then each level's run of the tile goes out
// to consecutive addresses (one coalesced write per run instead of one
// scattered write per range), the range fields read back from the tile just
// loaded (L1 / L2).  Same tiles as digit_offsets.
struct PlaceSmem {
    uint16_t lidx[RADIX_TILE];
    uint8_t dig[RADIX_TILE];
    uint32_t wcnt[(RADIX_THREADS / 32) * RADIX_BINS];
    uint32_t dstart[RADIX_BINS];
    uint32_t gbase[RADIX_BINS];
    uint32_t wbuf[33];
};
__global__ void __launch_bounds__(RADIX_THREADS) k_level_place(LevelDigit digit, const int64_t *__restrict__ start,
                                                               const int64_t *__restrict__ end,
                                                               const uint32_t *__restrict__ op, int64_t n,
                                                               const uint32_t *__restrict__ offs, int64_t ntiles,
                                                               int64_t *__restrict__ ls, int64_t *__restrict__ le,
                                                               uint32_t *__restrict__ li) {
    pdl_wait();
    __shared__ PlaceSmem S;
    const unsigned w = threadIdx.x >> 5, lane = lane_id();
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) S.wcnt[i] = 0;
    __syncthreads();
    const int64_t tile0 = (int64_t)blockIdx.x * RADIX_TILE;
    const int64_t base = tile0 + w * (RADIX_TILE / 8);
    unsigned dg[RADIX_ITEMS];
    uint32_t rank[RADIX_ITEMS];
    const unsigned lt = lanemask_lt();
    unsigned peers[RADIX_ITEMS];
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {        // digits and peer groups first: independent
        const int64_t i = base + it * 32 + lane;
        const unsigned d = i < n ? digit(i) : (unsigned)RADIX_BINS;
        peers[it] = warp_peers8(d, d < RADIX_BINS);
        dg[it] = d;
    }
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const unsigned d = dg[it];
        const unsigned before = d < RADIX_BINS ? S.wcnt[w * RADIX_BINS + d] : 0u;
        __syncwarp();
        if (d < RADIX_BINS && (peers[it] & lt) == 0) S.wcnt[w * RADIX_BINS + d] = before + __popc(peers[it]);
        __syncwarp();
        rank[it] = before + __popc(peers[it] & lt);
    }
    __syncthreads();
    uint32_t tot;
    {
        // RADIX_THREADS == RADIX_BINS: thread d owns digit d
        const unsigned d = threadIdx.x;
        uint32_t sum = 0;
#pragma unroll
        for (int q = 0; q < RADIX_THREADS / 32; ++q) {
            const uint32_t x = S.wcnt[q * RADIX_BINS + d];
            S.wcnt[q * RADIX_BINS + d] = sum;
            sum += x;
        }
        tot = sum;
    }
    const uint32_t ds = block_exclusive_scan<uint32_t>(tot, S.wbuf, (uint32_t *)nullptr);
    S.dstart[threadIdx.x] = ds;
    S.gbase[threadIdx.x] = offs[(int64_t)threadIdx.x * ntiles + blockIdx.x];
    __syncthreads();
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane;
        const unsigned d = dg[it];
        if (d < RADIX_BINS) {
            const uint32_t p = S.dstart[d] + S.wcnt[w * RADIX_BINS + d] + rank[it];
            S.lidx[p] = (uint16_t)(i - tile0);
            S.dig[p] = (uint8_t)d;
        }
    }
    __syncthreads();
    const int cnt = (int)(n - tile0 < RADIX_TILE ? n - tile0 : RADIX_TILE);
    constexpr int U = 4;                    // entries per thread per round, loads issued together
    for (int j0 = threadIdx.x; j0 < cnt; j0 += RADIX_THREADS * U) {
        uint32_t r[U];
        long long sv[U], ev[U];
        uint32_t ov[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int j = j0 + u * RADIX_THREADS;
            const int64_t i = tile0 + (j < cnt ? S.lidx[j] : 0);
            r[u] = digit.perm ? digit.perm[i] : (uint32_t)i;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            sv[u] = start[r[u]];
            ev[u] = end[r[u]];
            ov[u] = op[r[u]];
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int j = j0 + u * RADIX_THREADS;
            if (j >= cnt) continue;
            const unsigned d = S.dig[j];
            const int64_t o = (int64_t)S.gbase[d] + (j - S.dstart[d]);
            ls[o] = sv[u];
            le[o] = ev[u];
            li[o] = r[u] | (kind_of(ov[u]) << 30);
        }
    }
}

// Laminar checks over level positions: adjacent pairs of a level, and the
// parent of every range at depth > 0 (the last range of level (s, d-1) that
// starts no later; it must end no earlier).  A thread takes VL_PER
// consecutive positions: starts do not decrease along a level, so the parent
// is searched once and then followed forward.
constexpr int VL_PER = 8;
__global__ void k_validate_levels(const uint8_t *__restrict__ stream, const uint8_t *__restrict__ depth,
                                  const int64_t *__restrict__ ls, const int64_t *__restrict__ le,
                                  const uint32_t *__restrict__ li, const uint32_t *__restrict__ lvl_off, int64_t n,
                                  DevStatus *st) {
    pdl_wait();
    bool err = false, fix = false;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x * VL_PER;
    for (int64_t i0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * VL_PER; i0 < n; i0 += stride) {
        const int64_t i1 = i0 + VL_PER < n ? i0 + VL_PER : n;
        int64_t lend = -1, plo = 0, phi = 0, pp = 0;
        uint32_t d = 0;
        bool have_parent = false;
        long long a = ls[i0], b = le[i0];
        for (int64_t i = i0; i < i1; ++i) {
            if (i >= lend) {                     // the level of position i
                const uint32_t r = li[i] & 0x3FFFFFFFu;
                const uint32_t L = (uint32_t)stream[r] * 32u + depth[r];
                d = depth[r];
                lend = lvl_off[L + 1];
                if (d > 0) { plo = lvl_off[L - 1]; phi = lvl_off[L]; }
                have_parent = false;
            }
            long long a2 = 0, b2 = 0;
            if (i + 1 < n) { a2 = ls[i + 1]; b2 = le[i + 1]; }
            if (i + 1 < lend) {
                if (a2 == a && b2 < b) fix = true;
                else if (b > a2) err = true;
            }
            if (d > 0) {
                if (!have_parent) {              // last parent-level position with start <= a
                    int64_t x = plo, y = phi;
                    while (x < y) {
                        const int64_t m = (x + y) >> 1;
                        if (ls[m] <= a) x = m + 1; else y = m;
                    }
                    pp = x - 1;
                    have_parent = true;
                } else {
                    while (pp + 1 < phi && ls[pp + 1] <= a) ++pp;
                }
                if (pp < plo || le[pp] < b) err = true;
            }
            a = a2;
            b = b2;
        }
    }
    if (__any_sync(0xffffffffu, fix) && lane_id() == 0) set_flag(st, F_LEVEL_FIXUP);
    if (__any_sync(0xffffffffu, err) && lane_id() == 0) set_err(st, ERR_NOT_NESTED);
}

// ------------------------------------------------------------------ per-stream tiles
// The enclosure answers kernels stream by stream.  psk holds every kernel
// index regrouped by stream: a stable partition of the time-ordered kernels,
// so each stream's kernels are in time order, streams one after another
// (stream s from koff[s]).  Each stream's run is cut into tiles of EN_TILE
// kernels; tile r of stream s has the stream-major index u = toff[s] + r.
// Tiles are launched round-robin over the streams (tile r of every stream
// before tile r + 1 of any), so the tiles in flight cover one window of time
// and their gathers of start times and scattered result writes share sectors
// in L2.
constexpr int EN_THREADS = 128;
constexpr int EN_PER = 16;                        // consecutive kernels one thread sweeps
constexpr int EN_TILE = EN_THREADS * EN_PER;      // kernels of one stream per tile
constexpr int EN_WIN = 3072;                      // staged range entries per tile
constexpr int EN_RD = 8;                          // depths whose sweep state stays in registers

// The stream of the kernel at time position i (as its compact id: streams
// with kernels numbered in order), and its place in psk.
struct TimeStreamDigit {
    const uint8_t *stream;
    const uint32_t *korder;     // time order, NULL = array order
    const uint8_t *scmap;       // [256] compact id of a stream with kernels
    __device__ __forceinline__ unsigned operator()(int64_t i) const {
        return scmap[stream[korder ? korder[i] : (uint32_t)i]];
    }
};
// The stream of kernel i in array order (the kernels in time order).
struct ArrayStreamDigit {
    const uint8_t *stream;
    __device__ __forceinline__ unsigned operator()(int64_t i) const { return stream[i]; }
};
struct PlaceByStream {
    const uint32_t *korder;
    uint32_t *psk;
    __device__ __forceinline__ unsigned operator()(int64_t i, uint32_t dest, unsigned) const {
        psk[dest] = korder ? korder[i] : (uint32_t)i;
        return 0u;
    }
    __device__ __forceinline__ void done(unsigned) const {}
};

// Window of every (tile, depth): P[u * 32 + d] = (last position of level
// (s, d) with start <= the tile's first time, last position with start <= its
// last time), relative to the level's start, -1 for none.  Lane d of a warp
// takes depth d of one tile.  The warp also places the tile in the launch
// order: tile u = toff[s] + r goes to
//   sum over streams q of min(tiles of q, r)  +  #{q < s : tiles of q > r},
// tinfo[position] = s | r << 8.
__global__ void k_stream_windows(const int64_t *__restrict__ ls, const uint32_t *__restrict__ lvl_off,
                                 const uint8_t *__restrict__ ndep, const uint32_t *__restrict__ toff,
                                 const uint32_t *__restrict__ koff, const uint32_t *__restrict__ kcnt,
                                 const uint32_t *__restrict__ psk, const int64_t *__restrict__ k_start, int64_t nt,
                                 int2 *__restrict__ P, uint32_t *__restrict__ tinfo) {
    pdl_wait();
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < nt * 32; q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t u = q >> 5;
        const int d = (int)(q & 31);
        int lo = 0, hi = 256;
        while (hi - lo > 1) {
            const int m = (lo + hi) >> 1;
            if (toff[m] <= (uint32_t)u) lo = m; else hi = m;
        }
        const int sid = lo;
        {
            // the tile's launch position: each lane adds the terms of eight streams
            const uint32_t r = (uint32_t)u - toff[sid];
            uint32_t p = 0;
            for (int qs = d; qs < 256; qs += 32) {
                const uint32_t c = toff[qs + 1] - toff[qs];
                p += (c < r ? c : r) + (qs < sid && c > r ? 1u : 0u);
            }
            p = warp_sum<uint32_t>(p);
            if (d == 0) tinfo[p] = (uint32_t)sid | (r << 8);
        }
        if (d >= ndep[sid]) continue;
        const int64_t pos0 = (u - toff[sid]) * (int64_t)EN_TILE;
        const int64_t cnt = (int64_t)kcnt[sid] - pos0 < EN_TILE ? (int64_t)kcnt[sid] - pos0 : EN_TILE;
        const long long tf = k_start[psk[koff[sid] + pos0]], tl = k_start[psk[koff[sid] + pos0 + cnt - 1]];
        const int64_t L0 = lvl_off[sid * 32 + d], L1 = lvl_off[sid * 32 + d + 1];
        int64_t x = L0, y = L1;                    // first position with start > tf
        while (x < y) {
            const int64_t m = (x + y) >> 1;
            if (ls[m] <= tf) x = m + 1; else y = m;
        }
        const int64_t a = x;
        y = L1;                                    // first position with start > tl (at or after a)
        while (x < y) {
            const int64_t m = (x + y) >> 1;
            if (ls[m] <= tl) x = m + 1; else y = m;
        }
        P[q] = make_int2((int)(a - L0 - 1), (int)(x - L0 - 1));
    }
}

struct EncArgs {
    const int64_t *k_start;
    const uint32_t *psk, *tinfo, *toff, *koff, *kcnt;
    const uint8_t *ndep;
    const int64_t *ls, *le;
    const uint32_t *li;
    const uint32_t *lvl_off;    // [LEVELS + 1]
    const int2 *P;              // [tiles * 32]
    int32_t *out_range;
    uint8_t *out_nop;
};

struct EncSmem {
    uint32_t ws[EN_WIN];        // staged start, relative to the tile's first time (+1, clamped)
    uint32_t we[EN_WIN];        // staged end, same encoding
    uint32_t wi[EN_WIN];        // staged lvl_info
    int woff[32], wcnt[32];     // per depth: first staged entry and count
    int wlev[32];               // per depth: level position of the window's first entry
    int nwin;
};

__device__ __forceinline__ uint32_t rel32(long long x, long long base) {
    long long v = x - base + 1;
    return v <= 0 ? 0u : (v >= 0xFFFFFFFFll ? 0xFFFFFFFFu : (uint32_t)v);
}

// Algorithm 2's walk over one depth's representative, outward-in: a
// structural range resets the collection (everything above it is beyond the
// cut), an operator becomes the innermost answer and counts, a non-op range
// is passed over.
__device__ __forceinline__ void walk_step(uint32_t info, int32_t &ans, int &nop) {
    const uint32_t kind = info >> 30;
    if (kind == KIND_STRUCT) { ans = -1; nop = 0; }
    else if (kind == KIND_OP) { ans = (int32_t)(info & 0x3FFFFFFFu); nop++; }
}

// One tile of one stream.  Thread t sweeps the tile's kernels
// [t * EN_PER, (t + 1) * EN_PER) in time order, keeping per depth (the first
// EN_RD in registers) the last staged range starting at or before the
// current kernel: its position, end and info, and the next range's start.  A
// depth is searched once at the thread's first kernel and afterwards moves
// only when the next start is passed, so a kernel usually costs one
// comparison per depth.  The walk over the tracked depths runs for every
// kernel without branches (threads of a warp stay together; redoing it only
// when something changed saves less than the divergence costs); deeper
// levels are searched when the walk reaches them.  A tile whose windows outgrow the
// staging, or whose kernels span 2^32 ns or more (relative times no longer
// fit), searches the global level lists instead.
__global__ void __launch_bounds__(EN_THREADS) k_enclose(EncArgs A) {
    pdl_wait();
    __shared__ EncSmem S;
    const uint32_t info = A.tinfo[blockIdx.x];
    const int sid = (int)(info & 0xFFu);
    const uint32_t r = info >> 8;
    const int64_t u = A.toff[sid] + r;
    const int64_t pos0 = (int64_t)r * EN_TILE;
    const int cnt = (int)((int64_t)A.kcnt[sid] - pos0 < EN_TILE ? (int64_t)A.kcnt[sid] - pos0 : EN_TILE);
    const uint32_t *tk = A.psk + A.koff[sid] + pos0;         // the tile's kernels in time order
    const int nd = A.ndep[sid];
    const long long tbase = A.k_start[tk[0]], tlast = A.k_start[tk[cnt - 1]];
    const unsigned lane = lane_id(), warp = threadIdx.x >> 5;
    if (warp == 0) {
        const int d = (int)lane;
        int c = 0, first = 0;
        if (d < nd) {
            const int2 w = A.P[u * 32 + d];
            first = w.x < 0 ? 0 : w.x;
            c = w.y < 0 ? 0 : w.y - first + 1;
        }
        const int incl = warp_inclusive_scan(c);
        S.woff[d] = incl - c;
        S.wcnt[d] = c;
        S.wlev[d] = (d < nd ? (int)A.lvl_off[sid * 32 + d] : 0) + first;
        if (d == 31) S.nwin = incl;
    }
    __syncthreads();
    const bool slow = S.nwin > EN_WIN || (tlast - tbase) >= 0xFFFFFFF0ll;
    if (slow) {
        // global searches inside each depth's window
        for (int j = threadIdx.x; j < cnt; j += EN_THREADS) {
            const uint32_t k = tk[j];
            const long long T = A.k_start[k];
            int32_t ans = -1;
            int nop = 0;
            for (int d = 0; d < nd; ++d) {
                int64_t x = S.wlev[d], y = x + S.wcnt[d];
                const int64_t o = x;
                while (x < y) {
                    const int64_t m = (x + y) >> 1;
                    if (A.ls[m] <= T) x = m + 1; else y = m;
                }
                if (x == o || A.le[x - 1] < T) break;
                walk_step(A.li[x - 1], ans, nop);
            }
            A.out_range[k] = ans;
            if (A.out_nop) A.out_nop[k] = (uint8_t)nop;
        }
        return;
    }
    // stage the windows: one warp per depth, each depth's entries contiguous
    for (int d = (int)warp; d < nd; d += EN_THREADS / 32) {
        const int c = S.wcnt[d], o = S.woff[d];
        const int64_t g0 = S.wlev[d];
        for (int e = (int)lane; e < c; e += 32) {
            S.ws[o + e] = rel32(A.ls[g0 + e], tbase);
            S.we[o + e] = rel32(A.le[g0 + e], tbase);
            S.wi[o + e] = A.li[g0 + e];
        }
    }
    __syncthreads();
    constexpr uint32_t NONE_T = 0xFFFFFFFFu;
    const int j0 = (int)threadIdx.x * EN_PER;
    const int j1 = j0 + EN_PER < cnt ? j0 + EN_PER : cnt;
    if (j0 >= j1) return;
    int pos[EN_RD];                               // window position of the depth's range, -1 none
    uint32_t nxt[EN_RD], cend[EN_RD], cinf[EN_RD]; // next start; end and info of the range
    constexpr int B = 4;                          // kernels loaded per batch
    uint32_t kb[B];
    long long tb[B];
    auto load_batch = [&](int jb) {
#pragma unroll
        for (int v = 0; v < B; ++v) kb[v] = tk[jb + v < j1 ? jb + v : j0];
#pragma unroll
        for (int v = 0; v < B; ++v) tb[v] = A.k_start[kb[v]];
    };
    load_batch(j0);
    for (int jb = j0; jb < j1; jb += B) {
        uint32_t kc[B], tc[B];
#pragma unroll
        for (int v = 0; v < B; ++v) { kc[v] = kb[v]; tc[v] = rel32(tb[v], tbase); }
        if (jb + B < j1) load_batch(jb + B);      // the next batch in flight during this one
#pragma unroll
        for (int v = 0; v < B; ++v) {
            const int j = jb + v;
            if (j >= j1) break;
            const uint32_t T = tc[v];
            if (j == j0) {
#pragma unroll
                for (int d = 0; d < EN_RD; ++d) {
                    const int c = d < nd ? S.wcnt[d] : 0, o = d < nd ? S.woff[d] : 0;
                    int x = o, y = o + c;         // last window position with start <= T
                    while (x < y) {
                        const int m = (x + y) >> 1;
                        if (S.ws[m] <= T) x = m + 1; else y = m;
                    }
                    const int p = x - o - 1;
                    pos[d] = p;
                    nxt[d] = p + 1 < c ? S.ws[o + p + 1] : NONE_T;
                    cend[d] = p >= 0 ? S.we[o + p] : 0u;
                    cinf[d] = p >= 0 ? S.wi[o + p] : 0u;
                }
            } else {
#pragma unroll
                for (int d = 0; d < EN_RD; ++d) {
                    if (nxt[d] <= T) {            // a later range of this depth starts by T
                        const int c = S.wcnt[d], o = S.woff[d];
                        int p = pos[d] + 1;
                        while (p + 1 < c && S.ws[o + p + 1] <= T) ++p;
                        pos[d] = p;
                        nxt[d] = p + 1 < c ? S.ws[o + p + 1] : NONE_T;
                        cend[d] = S.we[o + p];
                        cinf[d] = S.wi[o + p];
                    }
                }
            }
            // the walk over the tracked depths, every kernel, without branches
            int32_t ans = -1;
            int nop = 0;
            bool alive = true;
#pragma unroll
            for (int d = 0; d < EN_RD; ++d) {
                alive = alive && d < nd && pos[d] >= 0 && cend[d] >= T;
                const uint32_t kind = cinf[d] >> 30;
                const bool st_d = alive && kind == KIND_STRUCT, op_d = alive && kind == KIND_OP;
                ans = st_d ? -1 : (op_d ? (int32_t)(cinf[d] & 0x3FFFFFFFu) : ans);
                nop = st_d ? 0 : nop + (op_d ? 1 : 0);
            }
            if (alive && nd > EN_RD) {
                for (int d = EN_RD; d < nd; ++d) {   // deeper levels: one search each
                    const int c = S.wcnt[d], o = S.woff[d];
                    int x = o, y = o + c;
                    while (x < y) {
                        const int m = (x + y) >> 1;
                        if (S.ws[m] <= T) x = m + 1; else y = m;
                    }
                    if (x == o || S.we[x - 1] < T) break;
                    walk_step(S.wi[x - 1], ans, nop);
                }
            }
            A.out_range[kc[v]] = ans;
            if (A.out_nop) A.out_nop[kc[v]] = (uint8_t)nop;
        }
    }
}

__global__ void k_fill_unattributed(int32_t *out_range, uint8_t *out_nop, int64_t n) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        out_range[i] = -1;
        if (out_nop) out_nop[i] = 0;
    }
}

// ------------------------------------------------------------------ host
static opattr_status status_from_err(unsigned err) {
    if (err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    if (err & ERR_DEPTH) return OPATTR_E_DEPTH;
    if (err & ERR_NOT_NESTED) return OPATTR_E_NOT_NESTED;
    if (err & ERR_TIMEOUT) return OPATTR_E_TIMEOUT;
    return OPATTR_OK;
}

opattr_status do_enclose(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, int32_t *out_range,
                         uint8_t *out_nop) {
    const int64_t K = kern->n, R = rng->n;
    if (K < 0 || R < 0 || R >= (1ll << 30) || K >= (1ll << 31)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->stream || !kern->start_ns || !out_range)) return OPATTR_E_INVALID_ARG;
    if (R > 0 && (!rng->stream || !rng->start_ns || !rng->end_ns || !rng->depth || !rng->op_id))
        return OPATTR_E_INVALID_ARG;

    // scratch: range sort (u64 keys x2, values x2), level arrays, tables,
    // kernel order, the stream partition of the kernels and its tile tables
    const int64_t nt_max = (K + EN_TILE - 1) / EN_TILE + 256;
    Need nd;
    nd.add<uint32_t>(LEVELS + 1 + 256).add<uint32_t>(LEVELS + 1).add<uint32_t>(radix_hist_elems(K));
    nd.add<uint64_t>(R).add<uint64_t>(R).add<uint32_t>(R).add<uint32_t>(R);
    const int64_t hist_n = std::max(radix_hist_elems(R), radix_hist_elems(K));
    const int64_t part_n = std::max<int64_t>(scan_scratch_elems(hist_n), scan_scratch_elems(LEVELS + 1));
    nd.add<uint32_t>(hist_n).add<uint32_t>(part_n).add<uint32_t>(hist_n).add<uint32_t>(part_n);
    nd.add<int64_t>(R).add<int64_t>(R).add<uint32_t>(R);
    nd.add<unsigned char>(STAGE_BYTES);
    nd.add<uint32_t>(K).add<uint32_t>(nt_max).add<int2>(nt_max * 32);
    const bool keep_order = c.in_join && K > 0;       // a join keeps the time order for its matching
    if (keep_order) nd.add<uint32_t>(K);
    size_t need = nd.bytes + kernel_order_scratch(K) + 4096;
    c.spec_ran = false;
    opattr_status st = ensure_arena(c, need);
    if (st) return st;
    if ((st = ensure_side(c))) return st;
    Arena a(c);
    uint32_t *kept_order = keep_order ? a.take<uint32_t>(K) : nullptr;     // first: the start of the arena
    if ((st = reset_status(c))) return st;

    // level histogram [LEVELS] and kernels per stream [256], zeroed together
    uint32_t *level_hist = a.take<uint32_t>(LEVELS + 1 + 256);
    uint32_t *kstream = level_hist + LEVELS + 1;
    uint32_t *lvl_off = a.take<uint32_t>(LEVELS + 1);
    uint32_t *part = a.take<uint32_t>(part_n), *part2 = a.take<uint32_t>(part_n);
    uint32_t *ktile = a.take<uint32_t>(radix_hist_elems(K));     // per tile, kernels of each stream
    if (!level_hist || !lvl_off || !part || !part2 || !ktile) return OPATTR_E_OOM;
    cudaMemsetAsync(level_hist, 0, sizeof(uint32_t) * (LEVELS + 1 + 256), c.stream);
    // the ranges' checks and level histogram on the side stream, beside the
    // kernels' order check; the level offsets and the stream counts come back
    // with the status: one synchronisation for all
    stream_after(c.side, c.stream, c.ev_fork);
    {
        OnStream on(c, c.side);
        if (R > 0)
            launch(c, "check_ranges", k_check_ranges, dim3(grid_for(R, RCHK_THREADS * RCHK_ITEMS)),
                   dim3(RCHK_THREADS), 0, rng->stream, rng->start_ns, rng->end_ns, rng->depth, R, level_hist,
                   c.d_status);
        scan_exclusive_u32(c, level_hist, lvl_off, LEVELS + 1, part2, nullptr);
    }
    check_kernel_order(c, kern->stream, kern->start_ns, K, kstream, ktile);
    stream_after(c.stream, c.side, c.ev_join);
    {
        // the level offsets and the stream counts come back with the status
        const SmallCopy back[2] = {{c.h_levels, lvl_off, sizeof(uint32_t) * (LEVELS + 1)},
                                   {c.h_levels + LEVELS + 1, kstream, sizeof(uint32_t) * 256}};
        if ((st = read_status(c, 2, back))) return st;
    }
    if ((st = status_from_err(c.h_status->err))) return st;
    const bool k_sorted = !(c.h_status->flags & F_K_UNSORTED);
    const bool r_sorted = !(c.h_status->flags & F_R_UNSORTED);
    c.enclose_k_sorted = k_sorted ? 1 : 0;
    const long long rmin = c.h_status->mm[MM_RSTART_MIN], rmax = c.h_status->mm[MM_REND_MAX];
    const long long kmin = c.h_status->mm[MM_KSTART_MIN], kmax = c.h_status->mm[MM_KSTART_MAX];
    if (K > 0 && (kmax - kmin) >= (1ll << 55)) return OPATTR_E_INVALID_ARG;

    if (R == 0) {
        if (K > 0)
            launch(c, "fill_unattributed", k_fill_unattributed, dim3(grid_for(K, 256, 65535)), dim3(256), 0, out_range,
                   out_nop, K);
        return read_status(c);
    }

    // ---- host-built tables, sent with one copy from pinned staging: level of
    // each compact level (u16 [LEVELS]), first compact level of a stream
    // (u16 [256]), levels of a stream (u8 [256]), compact id of a level
    // (u8 [LEVELS], at most 256 levels), and per stream its first place in
    // the stream partition, its kernels and its first tile (u32 [256],
    // [256], [257])
    constexpr size_t ST_LOC = 0, ST_CBASE = ST_LOC + 2 * LEVELS, ST_NDEP = ST_CBASE + 2 * 256,
                     ST_CMAP = ST_NDEP + 256, ST_KOFF = ST_CMAP + LEVELS, ST_KCNT = ST_KOFF + 4 * 256,
                     ST_TOFF = ST_KCNT + 4 * 256, ST_SCMAP = ST_TOFF + 4 * 257, ST_END = ST_SCMAP + 256;
    static_assert(ST_END <= STAGE_BYTES, "staging too small");
    const uint32_t *off = c.h_levels;
    const uint32_t *kcnt_h = c.h_levels + LEVELS + 1;
    uint16_t *level_of_compact = reinterpret_cast<uint16_t *>(c.h_stage + ST_LOC);
    uint16_t *cbase = reinterpret_cast<uint16_t *>(c.h_stage + ST_CBASE);
    uint8_t *ndep = c.h_stage + ST_NDEP;
    uint8_t *cmap = c.h_stage + ST_CMAP;
    uint32_t *koff_h = reinterpret_cast<uint32_t *>(c.h_stage + ST_KOFF);
    uint32_t *kcnt_s = reinterpret_cast<uint32_t *>(c.h_stage + ST_KCNT);
    uint32_t *toff_h = reinterpret_cast<uint32_t *>(c.h_stage + ST_TOFF);
    uint8_t *scmap = c.h_stage + ST_SCMAP;
    int nl = 0;
    for (int s = 0; s < 256; ++s) {
        cbase[s] = (uint16_t)nl;
        int n = 0;
        while (n < 32 && off[s * 32 + n + 1] > off[s * 32 + n]) {
            level_of_compact[nl++] = (uint16_t)(s * 32 + n);
            n++;
        }
        ndep[s] = (uint8_t)n;
    }
    memset(cmap, 0, LEVELS);
    for (int l = 0; l < nl && l < 256; ++l) cmap[level_of_compact[l]] = (uint8_t)l;
    uint32_t kacc = 0, tacc = 0;
    int nks = 0;                                  // streams with kernels
    for (int s = 0; s < 256; ++s) {
        scmap[s] = (uint8_t)nks;
        nks += kcnt_h[s] > 0;
        koff_h[s] = kacc;
        kcnt_s[s] = kcnt_h[s];
        toff_h[s] = tacc;
        kacc += kcnt_h[s];
        tacc += (kcnt_h[s] + EN_TILE - 1) / EN_TILE;
    }
    toff_h[256] = tacc;
    const int64_t NT = tacc;

    uint64_t *rk0 = a.take<uint64_t>(R), *rk1 = a.take<uint64_t>(R);
    uint32_t *rv0 = a.take<uint32_t>(R), *rv1 = a.take<uint32_t>(R);
    uint32_t *hist = a.take<uint32_t>(hist_n), *hist2 = a.take<uint32_t>(hist_n);
    int64_t *ls = a.take<int64_t>(R), *le = a.take<int64_t>(R);
    uint32_t *li = a.take<uint32_t>(R);
    unsigned char *d_stage = a.take<unsigned char>(ST_END);
    uint32_t *psk = a.take<uint32_t>(K), *tinfo = a.take<uint32_t>(NT);
    int2 *P = a.take<int2>(NT * 32);
    if (!rk0 || !rk1 || !rv0 || !rv1 || !hist || !hist2 || !ls || !le || !li || !d_stage || !psk || !tinfo || !P)
        return OPATTR_E_OOM;
    const uint8_t *d_ndep = d_stage + ST_NDEP;
    const uint8_t *d_cmap = d_stage + ST_CMAP;
    const uint32_t *d_koff = reinterpret_cast<const uint32_t *>(d_stage + ST_KOFF);
    const uint32_t *d_kcnt = reinterpret_cast<const uint32_t *>(d_stage + ST_KCNT);
    const uint32_t *d_toff = reinterpret_cast<const uint32_t *>(d_stage + ST_TOFF);
    const uint8_t *d_scmap = d_stage + ST_SCMAP;
    if ((st = copy_small(c, d_stage, c.h_stage, ST_END, cudaMemcpyHostToDevice))) return st;
    // the level lists (below) may start on the side stream from here
    stream_after(c.side, c.stream, c.ev_fork);

    // ---- kernel time order, then the kernels partitioned by stream
    uint32_t *korder = nullptr;
    if (!k_sorted && K > 0) {
        // keyed by the compact ids of the streams with kernels
        korder = kernel_time_order(c, a, kern->stream, kern->start_ns, K, d_scmap, bits_for((uint64_t)(nks - 1)));
        if (!korder) return OPATTR_E_OOM;
        if (kept_order) {
            cudaMemcpyAsync(kept_order, korder, sizeof(uint32_t) * K, cudaMemcpyDeviceToDevice, c.stream);
            c.join_korder = kept_order;
            c.arena_keep = (sizeof(uint32_t) * (size_t)K + 255) & ~(size_t)255;
        }
    }
    if (K > 0 && nl > 0 && k_sorted) {
        // in time order already: the order check's tile counts are the
        // partition's histogram (stream ids as digits)
        // (rows past the last stream with kernels hold only zeros: not scanned)
        const int64_t ntk = (K + RADIX_TILE - 1) / RADIX_TILE;
        int rows = 0;
        for (int q = 0; q < 256; ++q)
            if (kcnt_h[q] > 0) rows = q + 1;
        scan_exclusive_u32(c, ktile, hist, ntk * rows, part, nullptr);
        digit_rank(c, "stream_place", ArrayStreamDigit{kern->stream}, K, hist, PlaceByStream{nullptr, psk});
    } else if (K > 0 && nl > 0) {
        const TimeStreamDigit dg{kern->stream, korder, d_scmap};
        const uint32_t *offs = digit_offsets(c, dg, K, hist, part, nks);
        digit_rank(c, "stream_place", dg, K, offs, PlaceByStream{korder, psk});
    }

    // ---- level lists, their validation, the windows and the enclosure, without
    // a synchronisation in between: a failed validation is reported at the end
    // (the enclosure reads only positions found by searches inside the level
    // lists, so non-laminar ranges give wrong answers but no stray access).
    // If ranges with equal starts were not in (start, end, index) order within
    // a level, the whole pass runs again on fully sorted ranges.  The level
    // lists and their validation run on the side stream, beside the stream
    // partition (their own scratch: hist2, part2); the windows wait for the
    // lists, the status read for the validation.
    const unsigned g = grid_for(R, 256, 65535);
    for (int attempt = 0; attempt < 2; ++attempt) {
        const bool full_sort = !r_sorted || attempt > 0;
        if (attempt > 0) stream_after(c.side, c.stream, c.ev_fork);
        {
            OnStream on(c, c.side);
            uint32_t *perm = nullptr;     // range indices in the order of the level sort
            if (full_sort) {
                // (start, end, index) order within every level of laminar
                // ranges: one stable sort on (start, longer than zero)
                uint64_t *ko;
                const int bits = bits_for((uint64_t)(rmax - rmin)) + 1;
                launch(c, "range_time_key", k_range_start_key, dim3(g), dim3(256), 0, rng->start_ns, rng->end_ns, R,
                       rmin, rk0);
                radix_sort_pairs<uint64_t>(c, rk0, rv0, rk1, rv1, R, bits, true, hist2, part2, &ko, &perm);
            }
            if (nl <= 256) {
                // stable partition by compact level id, ranges written in place
                const LevelDigit dg{rng->stream, rng->depth, d_cmap, perm};
                const uint32_t *offs = digit_offsets(c, dg, R, hist2, part2, nl);
                const int64_t ntiles = (R + RADIX_TILE - 1) / RADIX_TILE;
                launch(c, "level_place", k_level_place, dim3((unsigned)ntiles), dim3(RADIX_THREADS), 0, dg,
                       rng->start_ns, rng->end_ns, rng->op_id, R, offs, ntiles, ls, le, li);
            } else {
                // stable partition by level key (13 bits)
                uint32_t *lk0 = reinterpret_cast<uint32_t *>(rk0), *lk1 = reinterpret_cast<uint32_t *>(rk1);
                uint32_t *va = perm ? perm : rv0;
                uint32_t *vb = perm == rv0 ? rv1 : (perm == rv1 ? rv0 : rv1);
                launch(c, "level_keys", k_level_keys, dim3(g), dim3(256), 0, rng->stream, rng->depth,
                       (const uint32_t *)perm, R, lk0);
                uint32_t *ko32, *lperm;
                radix_sort_pairs<uint32_t>(c, lk0, va, lk1, vb, R, 13, perm == nullptr, hist2, part2, &ko32, &lperm);
                launch(c, "level_gather", k_level_gather, dim3(g), dim3(256), 0, rng->start_ns, rng->end_ns,
                       rng->op_id, (const uint32_t *)lperm, R, ls, le, li);
            }
            cudaEventRecord(c.ev_join, c.side);           // the level lists are in place
            launch(c, "validate_levels", k_validate_levels, dim3(grid_for(R, 256 * VL_PER, 65535)), dim3(256), 0,
                   rng->stream, rng->depth, (const int64_t *)ls, (const int64_t *)le, (const uint32_t *)li,
                   (const uint32_t *)lvl_off, R, c.d_status);
            // within a join: the matching's identity pairing, beside the enclosure
            if (c.spec_k > 0) {
                launch_identity_match(c, c.spec_kname, c.spec_nname, c.spec_k, c.spec_idx, c.spec_kind);
                c.spec_ran = true;
            }
            cudaEventRecord(c.ev_join2, c.side);          // and checked
        }
        cudaStreamWaitEvent(c.stream, c.ev_join, 0);
        if (K > 0 && nl == 0)
            launch(c, "fill_unattributed", k_fill_unattributed, dim3(grid_for(K, 256, 65535)), dim3(256), 0, out_range,
                   out_nop, K);
        if (K > 0 && nl > 0) {
            launch(c, "stream_windows", k_stream_windows, dim3(grid_for(NT * 32, 256, 65535)), dim3(256), 0,
                   (const int64_t *)ls, (const uint32_t *)lvl_off, d_ndep, d_toff, d_koff, d_kcnt,
                   (const uint32_t *)psk, kern->start_ns, NT, P, tinfo);
            EncArgs A;
            A.k_start = kern->start_ns;
            A.psk = psk;
            A.tinfo = tinfo;
            A.toff = d_toff;
            A.koff = d_koff;
            A.kcnt = d_kcnt;
            A.ndep = d_ndep;
            A.ls = ls;
            A.le = le;
            A.li = li;
            A.lvl_off = lvl_off;
            A.P = P;
            A.out_range = out_range;
            A.out_nop = out_nop;
            launch(c, "enclose", k_enclose, dim3((unsigned)NT), dim3(EN_THREADS), 0, A);
        }
        cudaStreamWaitEvent(c.stream, c.ev_join2, 0);
        if (c.defer_status && k_sorted && !full_sort) {
            // the status is read with the aggregation's, which the join checks
            c.enclose_pending = true;
            return OPATTR_OK;
        }
        if ((st = read_status(c))) return st;
        if (!full_sort && (c.h_status->flags & F_LEVEL_FIXUP)) {
            // equal starts out of (start, end) order within a level: the
            // nesting checks above saw a level list out of order, so their
            // verdict does not count; the pass on fully sorted ranges decides
            c.h_status->flags &= ~F_LEVEL_FIXUP;
            c.h_status->err = 0;
            cudaMemsetAsync(c.d_status, 0, 2 * sizeof(unsigned), c.stream);   // err and flags
            continue;
        }
        if ((st = status_from_err(c.h_status->err))) return st;
        // after the sort, equal starts out of (start, end) order in a level
        // are two longer ranges with one start: overlapping, not laminar
        if (c.h_status->flags & F_LEVEL_FIXUP) return OPATTR_E_NOT_NESTED;
        return OPATTR_OK;
    }
    return OPATTR_E_CUDA;
}

}  // namespace opattr
