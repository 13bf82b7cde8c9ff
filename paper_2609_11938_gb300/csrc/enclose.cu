// enclose.cu -- Algorithm 2 (NVTX enclosure attribution, Sec. 3.5) on the GPU.
//
// Data layout.  Ranges are regrouped into per-(stream, depth) level lists,
// each in (start, end, index) order: lvl_start / lvl_end (i64) and lvl_info
// (u32: range index in the low 30 bits, kind in the top 2: 0 operator,
// 1 non-op, 2 structural).  lvl_off[level] gives the list bounds, level =
// stream * 32 + depth.  Within a level ranges are disjoint or touching, so
// "the last range with start <= T" is the only one that can contain T.
//
// Kernels are taken in time order, in tiles of ENC_TILE.  A window table
// P[tile][level] (last level position with start <= the tile's first T) bounds,
// per level, the ranges a tile can hit; the enclosure kernel stages those
// windows in shared memory as 32-bit times relative to the tile start and
// answers each kernel by one search per depth, walking depths outward-in
// (0, 1, ...) until a depth has no containing range.  The walk state needs no
// stack: a structural range resets the collection (everything above it is
// beyond the cut); an operator becomes the innermost answer and counts;
// a non-op range is passed over.
#include <algorithm>

#include "sort.cuh"
#include "util.cuh"

namespace opattr {

constexpr int LEVELS = N_LEVELS;
constexpr int ENC_THREADS = 256;
constexpr int ENC_TILE = 2048;          // kernels per tile
// Shared-memory capacities: staged range entries and active (stream, depth)
// levels per tile.  With few levels a compact layout (and 64 registers)
// keeps four blocks per SM; a tile that outgrows it is deferred to the wide
// layout, which handles any tile (overflowing ones by global searches).
constexpr int ENC_WIN_SMALL = 1024, ENC_ACT_SMALL = 256;
constexpr int ENC_WIN_WIDE = 3072, ENC_ACT_WIDE = 2048;
constexpr int ENC_CHUNK = ENC_TILE / ENC_THREADS;   // consecutive same-stream kernels per thread
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
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = perm ? perm[i] : i;
        keys[i] = (uint32_t)stream[r] * 32u + depth[r];
    }
}
__global__ void k_time_key(const int64_t *__restrict__ t, const uint32_t *__restrict__ perm, int64_t n,
                           long long tmin, uint64_t *__restrict__ keys) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t r = perm ? perm[i] : i;
        keys[i] = (uint64_t)(t[r] - tmin);
    }
}
__global__ void k_level_gather(const int64_t *__restrict__ start, const int64_t *__restrict__ end,
                               const uint32_t *__restrict__ op, const uint32_t *__restrict__ perm, int64_t n,
                               int64_t *__restrict__ ls, int64_t *__restrict__ le, uint32_t *__restrict__ li) {
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
    __shared__ PlaceSmem S;
    const unsigned w = threadIdx.x >> 5, lane = lane_id();
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) S.wcnt[i] = 0;
    __syncthreads();
    const int64_t tile0 = (int64_t)blockIdx.x * RADIX_TILE;
    const int64_t base = tile0 + w * (RADIX_TILE / 8);
    unsigned dg[RADIX_ITEMS];
    uint32_t rank[RADIX_ITEMS];
    const unsigned lt = lanemask_lt();
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane;
        const unsigned d = i < n ? digit(i) : (unsigned)RADIX_BINS;
        const unsigned peers = __match_any_sync(0xffffffffu, d);
        const unsigned before = d < RADIX_BINS ? S.wcnt[w * RADIX_BINS + d] : 0u;
        __syncwarp();
        if (d < RADIX_BINS && (peers & lt) == 0) S.wcnt[w * RADIX_BINS + d] = before + __popc(peers);
        __syncwarp();
        rank[it] = before + __popc(peers & lt);
        dg[it] = d;
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
// starts no later; it must end no earlier).
__global__ void k_validate_levels(const uint8_t *__restrict__ stream, const uint8_t *__restrict__ depth,
                                  const int64_t *__restrict__ ls, const int64_t *__restrict__ le,
                                  const uint32_t *__restrict__ li, const uint32_t *__restrict__ lvl_off, int64_t n,
                                  DevStatus *st) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t r = li[i] & 0x3FFFFFFFu;
        uint32_t s = stream[r], d = depth[r];
        uint32_t L = s * 32 + d;
        long long a = ls[i], b = le[i];
        if (i + 1 < (int64_t)lvl_off[L + 1]) {
            long long a2 = ls[i + 1], b2 = le[i + 1];
            if (a2 == a && b2 < b) set_flag(st, F_LEVEL_FIXUP);
            else if (b > a2) set_err(st, ERR_NOT_NESTED);
        }
        if (d > 0) {
            int64_t lo = lvl_off[L - 1], hi = lvl_off[L];
            int64_t x = lo, y = hi;               // first position with start > a
            while (x < y) {
                int64_t m = (x + y) >> 1;
                if (ls[m] <= a) x = m + 1; else y = m;
            }
            if (x == lo || le[x - 1] < b) set_err(st, ERR_NOT_NESTED);
        }
    }
}

// ------------------------------------------------------------------ window table
// P[t * nl + l] = (last position p of level l with lvl_start[p] <= b_t) - level
// start, or -1; b_t = start of the time-ordered kernel t*ENC_TILE for
// t < nt, and of the last kernel for t = nt.  The b_t do not decrease, so
// one thread takes `chunk` consecutive tiles of one level: a binary search
// for the first, then an exponential search forward from the previous
// answer for each next one (cost logarithmic in the entries passed, however
// unevenly a level's ranges fall between tiles).  Neighbouring threads take
// neighbouring levels, so the rows of P are written together.  Small tables
// take chunks of one tile (every search in parallel).
constexpr int WT_CHUNK = 16;
__device__ __forceinline__ long long tile_bound(const int64_t *k_start, const uint32_t *korder, int64_t K, int64_t nt,
                                                int64_t t) {
    const int64_t pos = t < nt ? t * ENC_TILE : K - 1;
    return k_start[korder ? korder[pos] : pos];
}
__global__ void k_window_table(const int64_t *__restrict__ ls, const uint32_t *__restrict__ lvl_off,
                               const uint16_t *__restrict__ level_of_compact, int nl,
                               const int64_t *__restrict__ k_start, const uint32_t *__restrict__ korder, int64_t K,
                               int64_t nt, int chunk, int32_t *__restrict__ P) {
    const int64_t nchunk = (nt + 1 + chunk - 1) / chunk;
    const int64_t total = nchunk * nl;
    for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t ch = q / nl;
        const int l = (int)(q - ch * nl);
        const uint32_t L = level_of_compact[l];
        const int64_t lo = lvl_off[L], hi = lvl_off[L + 1];
        const int64_t t0 = ch * chunk, t1 = t0 + chunk < nt + 1 ? t0 + chunk : nt + 1;
        int64_t x = lo;                       // first position with start > b (for the current tile)
        for (int64_t t = t0; t < t1; ++t) {
            const long long b = tile_bound(k_start, korder, K, nt, t);
            int64_t a2 = x, z = x;
            if (t > t0) {
                int64_t step = 1;
                while (z < hi && ls[z] <= b) {
                    a2 = z + 1;
                    z += step;
                    step <<= 1;
                }
                if (z > hi) z = hi;
            } else {
                z = hi;
            }
            while (a2 < z) {                  // first position in [a2, z) with start > b, else z
                const int64_t m = (a2 + z) >> 1;
                if (ls[m] <= b) a2 = m + 1; else z = m;
            }
            x = a2;
            P[t * nl + l] = (int32_t)(x - lo - 1);
        }
    }
}

// ------------------------------------------------------------------ enclosure
struct EncArgs {
    const uint8_t *k_stream;
    const int64_t *k_start;
    const uint32_t *korder;     // NULL = identity
    int64_t K;
    const int64_t *ls, *le;
    const uint32_t *li;
    const uint32_t *lvl_off;    // [LEVELS + 1]
    const int32_t *P;           // [(nt + 1) * nl]
    int nl;
    int64_t nt;
    const uint16_t *cbase;      // [256] first compact level of a stream
    const uint16_t *level_of_compact;   // [nl] level key (stream * 32 + depth) of a compact level
    const uint8_t *ndepth;      // [256] levels of a stream (depths 0 .. n-1)
    int32_t *out_range;
    uint8_t *out_nop;
    const uint32_t *tiles;      // tiles to process (deferred ones), or NULL for 0 .. nt-1
    const unsigned *ntiles;     // their count (device), with `tiles`
    uint32_t *deferred;         // compact-layout pass: tiles handed to the wide pass
    unsigned *ndeferred;
};

template <int WIN, int ACT>
struct EncSmem {
    uint32_t ws[WIN];               // staged start, relative to tile base (+1, clamped)
    uint32_t we[WIN];               // staged end, same encoding
    uint32_t wi[WIN];               // staged lvl_info
    uint16_t act_off[ACT];          // window offset of an active level
    uint16_t act_cnt[ACT];          // window length
    int32_t act_gpos[ACT];          // global level position of the window's first entry (-1 none)
    uint16_t sbase[256];            // first active slot of a present stream
    uint32_t kt[ENC_TILE];          // the tile's kernel times, relative to the tile base (+1, clamped)
    uint8_t ks[ENC_TILE];           // the tile's kernel streams
    uint16_t klist[ENC_TILE];       // tile positions grouped by stream
    uint16_t wcnt[ENC_THREADS / 32][256];
    uint16_t soff[257];
    uint32_t present[8];
    uint32_t wbuf[33];
    int slow;
    int nact, nwin;
};

__device__ __forceinline__ uint32_t rel32(long long x, long long base) {
    long long v = x - base + 1;
    return v <= 0 ? 0u : (v >= 0xFFFFFFFFll ? 0xFFFFFFFFu : (uint32_t)v);
}

// One tile.  DEFER: a tile that outgrows the layout is handed on (its index
// appended to A.deferred) instead of taking the global-search path.
template <int WIN, int ACT, bool DEFER>
__device__ __forceinline__ void enclose_tile(const EncArgs &A, EncSmem<WIN, ACT> &S, const int64_t t) {
    const int64_t pos0 = t * ENC_TILE;
    const int64_t cnt = A.K - pos0 < ENC_TILE ? A.K - pos0 : ENC_TILE;
    if (threadIdx.x < 8) S.present[threadIdx.x] = 0;
    __syncthreads();

    const long long tbase = A.k_start[A.korder ? A.korder[pos0] : pos0];
    {
        // all loads first, so they are in flight together
        constexpr int PER = ENC_TILE / ENC_THREADS;
        unsigned sv[PER];
        long long tv[PER];
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int j = u * ENC_THREADS + threadIdx.x;
            const int64_t p = pos0 + (j < cnt ? j : 0);
            const int64_t k = A.korder ? A.korder[p] : p;
            sv[u] = A.k_stream[k];
            tv[u] = A.k_start[k];
        }
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int j = u * ENC_THREADS + threadIdx.x;
            if (j < cnt) {
                S.ks[j] = (uint8_t)sv[u];
                S.kt[j] = rel32(tv[u], tbase);
                atomicOr(&S.present[sv[u] >> 5], 1u << (sv[u] & 31));
            }
        }
    }
    __syncthreads();

    // active levels: the levels of every stream present in the tile
    {
        const unsigned s = threadIdx.x;        // ENC_THREADS == 256 streams
        unsigned n = ((S.present[s >> 5] >> (s & 31)) & 1u) ? A.ndepth[s] : 0u;
        unsigned tot;
        unsigned off = block_exclusive_scan<unsigned>(n, S.wbuf, &tot);
        S.sbase[s] = (uint16_t)(off < ACT ? off : ACT);
        if (threadIdx.x == 0) S.nact = (int)tot;
        if (tot <= ACT && n) {
            const unsigned cb = A.cbase[s];
            for (unsigned d = 0; d < n; ++d) S.act_off[off + d] = (uint16_t)(cb + d);   // compact level, for now
        }
        __syncthreads();
        // window bounds of every active level, one thread per level
        if (tot <= ACT) {
            for (unsigned a = threadIdx.x; a < tot; a += ENC_THREADS) {
                const int l = S.act_off[a];
                const int32_t lo = A.P[t * A.nl + l], hi = A.P[(t + 1) * A.nl + l];
                const int32_t first = lo < 0 ? 0 : lo;
                int32_t c = hi - first + 1;
                if (hi < 0) c = 0;
                S.act_cnt[a] = (uint16_t)(c < 0xFFFF ? c : 0xFFFF);
                S.act_gpos[a] = (int32_t)(A.lvl_off[A.level_of_compact[l]] + first);
            }
        }
    }
    __syncthreads();
    // span of the tile: its last kernel (time order) minus its first
    const long long tlast = A.k_start[A.korder ? A.korder[pos0 + cnt - 1] : pos0 + cnt - 1];
    int slow = S.nact > ACT || (tlast - tbase) >= 0xFFFFFFF0ll;
    if (!slow) {
        // window offsets: exclusive scan of counts over active slots
        unsigned carry = 0;
        for (int b = 0; b < S.nact; b += ENC_THREADS) {
            int a = b + threadIdx.x;
            unsigned c = a < S.nact ? S.act_cnt[a] : 0u;
            unsigned tot;
            unsigned off = block_exclusive_scan<unsigned>(c, S.wbuf, &tot);
            if (a < S.nact) S.act_off[a] = (uint16_t)((carry + off) < 0xFFFF ? carry + off : 0xFFFF);
            carry += tot;
        }
        if (threadIdx.x == 0) S.nwin = (int)carry;
        __syncthreads();
        slow = S.nwin > WIN;
    }
    if (!slow) {
        // stage the windows: one thread per staged entry (its level found by a
        // search over the window offsets), so all loads of a round are in flight
        // together
        const int nact = S.nact, nwin = S.nwin;
        for (int e = threadIdx.x; e < nwin; e += ENC_THREADS) {
            int x = 0, y = nact;                   // last active level with offset <= e
            while (y - x > 1) {
                const int m = (x + y) >> 1;
                if (S.act_off[m] <= e) x = m; else y = m;
            }
            while (x + 1 < nact && S.act_off[x + 1] <= e && S.act_cnt[x] == 0) ++x;
            const int64_t g = S.act_gpos[x] + (e - S.act_off[x]);
            S.ws[e] = rel32(A.ls[g], tbase);
            S.we[e] = rel32(A.le[g], tbase);
            S.wi[e] = A.li[g];
        }
        // kernels grouped by stream, so a warp's lanes share windows and
        // loop trip counts
        block_group_by_key<ENC_THREADS, ENC_TILE / (ENC_THREADS / 32)>(
            256, [&](int j) -> unsigned { return j < cnt ? (unsigned)S.ks[j] : GROUP_NONE; }, &S.wcnt[0][0], 256,
            S.soff, S.klist, S.wbuf);
        // Each thread sweeps ENC_CHUNK consecutive kernels of one stream in
        // time order, keeping per depth (the first RD depths, in registers)
        // the last window range starting at or before the current kernel:
        // its position, end and info, and the start of the next one.  A depth
        // is searched once when the stream changes and afterwards moves only
        // when the next range's start is passed (positions only move
        // forward), so a kernel usually costs one comparison per depth.
        // The walk over the depths is redone only when a depth moved or a
        // range it found has ended; otherwise it would visit the same ranges
        // with the same results.
        constexpr int RD = 8;                     // depths whose state stays in registers
        constexpr uint32_t NONE_T = 0xFFFFFFFFu;
        int cur_s = -1, nd = 0, a0 = 0;
        int pos[RD];                              // window position of the depth's range, -1 none
        uint32_t nxt[RD], cend[RD], cinf[RD];     // next start; end and info of the range
#pragma unroll
        for (int d = 0; d < RD; ++d) pos[d] = -1, nxt[d] = NONE_T, cend[d] = 0, cinf[d] = 0;
        int32_t ans = -1;
        int nop = 0;
        bool redo = true;                         // the walk must be redone
        uint32_t min_end = 0;                     // earliest end among the ranges the walk went through
        for (int u = 0; u < ENC_CHUNK; ++u) {
            const int idx = threadIdx.x * ENC_CHUNK + u;
            if (idx >= cnt) break;
            const int j = S.klist[idx];
            const int64_t k = A.korder ? A.korder[pos0 + j] : pos0 + j;
            const int s = S.ks[j];
            const uint32_t T = S.kt[j];
            if (s != cur_s) {
                cur_s = s;
                nd = A.ndepth[s];
                a0 = S.sbase[s];
#pragma unroll
                for (int d = 0; d < RD; ++d) {
                    const int c = d < nd ? S.act_cnt[a0 + d] : 0, o = d < nd ? S.act_off[a0 + d] : 0;
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
                redo = true;
            } else {
#pragma unroll
                for (int d = 0; d < RD; ++d) {
                    if (nxt[d] <= T) {            // a later range of this depth starts by T
                        const int c = S.act_cnt[a0 + d], o = S.act_off[a0 + d];
                        int p = pos[d] + 1;
                        while (p + 1 < c && S.ws[o + p + 1] <= T) ++p;
                        pos[d] = p;
                        nxt[d] = p + 1 < c ? S.ws[o + p + 1] : NONE_T;
                        cend[d] = S.we[o + p];
                        cinf[d] = S.wi[o + p];
                        redo = true;
                    }
                }
                redo = redo || T > min_end;
            }
            if (redo) {
                ans = -1;
                nop = 0;
                bool alive = true;
                min_end = NONE_T;
#pragma unroll
                for (int d = 0; d < RD; ++d) {
                    if (alive && d < nd) {
                        if (pos[d] < 0 || cend[d] < T) {
                            alive = false;
                        } else {
                            min_end = min(min_end, cend[d]);
                            const uint32_t kind = cinf[d] >> 30;
                            if (kind == KIND_STRUCT) { ans = -1; nop = 0; }
                            else if (kind == KIND_OP) { ans = (int32_t)(cinf[d] & 0x3FFFFFFFu); nop++; }
                        }
                    }
                }
                bool deep = false;
                for (int d = RD; alive && d < nd; ++d) {   // deeper levels: one search each
                    deep = true;
                    const int c = S.act_cnt[a0 + d], o = S.act_off[a0 + d];
                    int x = o, y = o + c;
                    while (x < y) {
                        const int m = (x + y) >> 1;
                        if (S.ws[m] <= T) x = m + 1; else y = m;
                    }
                    if (x == o || S.we[x - 1] < T) break;
                    const uint32_t info = S.wi[x - 1];
                    const uint32_t kind = info >> 30;
                    if (kind == KIND_STRUCT) { ans = -1; nop = 0; }
                    else if (kind == KIND_OP) { ans = (int32_t)(info & 0x3FFFFFFFu); nop++; }
                }
                redo = deep;                      // deep levels are not tracked: search again next time
            }
            A.out_range[k] = ans;
            if (A.out_nop) A.out_nop[k] = (uint8_t)nop;
        }
        return;
    }
    if (DEFER) {                           // the wide pass takes this tile
        if (threadIdx.x == 0) A.deferred[atomicAdd(A.ndeferred, 1u)] = (uint32_t)t;
        return;
    }
    // slow tile: search the global level lists inside the window bounds
    for (int j = threadIdx.x; j < cnt; j += ENC_THREADS) {
        const int64_t p = pos0 + j;
        const int64_t k = A.korder ? A.korder[p] : p;
        const unsigned s = A.k_stream[k];
        const long long T = A.k_start[k];
        const int nd = A.ndepth[s];
        int32_t ans = -1;
        int nop = 0;
        for (int d = 0; d < nd; ++d) {
            int l = A.cbase[s] + d;
            int32_t lo = A.P[t * A.nl + l], hi = A.P[(t + 1) * A.nl + l];
            if (hi < 0) break;
            int64_t g0 = A.lvl_off[s * 32 + d];
            int64_t x = g0 + (lo < 0 ? 0 : lo), y = g0 + hi + 1, o = x;
            while (x < y) {
                int64_t m = (x + y) >> 1;
                if (A.ls[m] <= T) x = m + 1; else y = m;
            }
            if (x == o || A.le[x - 1] < T) break;
            uint32_t info = A.li[x - 1];
            uint32_t kind = info >> 30;
            if (kind == KIND_STRUCT) { ans = -1; nop = 0; }
            else if (kind == KIND_OP) { ans = (int32_t)(info & 0x3FFFFFFFu); nop++; }
        }
        A.out_range[k] = ans;
        if (A.out_nop) A.out_nop[k] = (uint8_t)nop;
    }
}

using EncSmemSmall = EncSmem<ENC_WIN_SMALL, ENC_ACT_SMALL>;
using EncSmemWide = EncSmem<ENC_WIN_WIDE, ENC_ACT_WIDE>;

// Compact layout, one tile per block, four blocks per SM; tiles that outgrow
// it are deferred to k_enclose_wide.
__global__ void __launch_bounds__(ENC_THREADS, 4) k_enclose(EncArgs A) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    enclose_tile<ENC_WIN_SMALL, ENC_ACT_SMALL, true>(A, *reinterpret_cast<EncSmemSmall *>(smem_raw), blockIdx.x);
}

// Wide layout: every tile (A.tiles NULL) or the deferred ones.
__global__ void __launch_bounds__(ENC_THREADS) k_enclose_wide(EncArgs A) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    EncSmemWide &S = *reinterpret_cast<EncSmemWide *>(smem_raw);
    const int64_t n = A.tiles ? (int64_t)*A.ntiles : A.nt;
    for (int64_t i = blockIdx.x; i < n; i += gridDim.x) {
        enclose_tile<ENC_WIN_WIDE, ENC_ACT_WIDE, false>(A, S, A.tiles ? (int64_t)A.tiles[i] : i);
        __syncthreads();                   // the next tile reuses the shared memory
    }
}

__global__ void k_fill_unattributed(int32_t *out_range, uint8_t *out_nop, int64_t n) {
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

    // scratch: range sort (u64 keys x2, values x2), level arrays, tables, kernel order
    const int64_t nt = (K + ENC_TILE - 1) / ENC_TILE;
    Need nd;
    nd.add<uint32_t>(LEVELS + 1).add<uint32_t>(LEVELS + 1);
    nd.add<uint64_t>(R).add<uint64_t>(R).add<uint32_t>(R).add<uint32_t>(R);
    const int64_t part_n = std::max<int64_t>(scan_scratch_elems(radix_hist_elems(R)), scan_scratch_elems(LEVELS + 1));
    nd.add<uint32_t>(radix_hist_elems(R)).add<uint32_t>(part_n);
    nd.add<int64_t>(R).add<int64_t>(R).add<uint32_t>(R);
    nd.add<unsigned char>(STAGE_BYTES);
    nd.add<int32_t>((nt + 1) * (int64_t)LEVELS).add<uint32_t>(nt).add<unsigned>(1);
    size_t need = nd.bytes + kernel_order_scratch(K) + 4096;
    opattr_status st = ensure_arena(c, need);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;

    uint32_t *level_hist = a.take<uint32_t>(LEVELS + 1);
    uint32_t *lvl_off = a.take<uint32_t>(LEVELS + 1);
    uint32_t *part = a.take<uint32_t>(part_n);
    if (!level_hist || !lvl_off || !part) return OPATTR_E_OOM;
    cudaMemsetAsync(level_hist, 0, sizeof(uint32_t) * (LEVELS + 1), c.stream);
    if (R > 0)
        launch(c, "check_ranges", k_check_ranges, dim3(grid_for(R, RCHK_THREADS * RCHK_ITEMS)), dim3(RCHK_THREADS), 0,
               rng->stream, rng->start_ns, rng->end_ns, rng->depth, R, level_hist, c.d_status);
    check_kernel_order(c, kern->stream, kern->start_ns, K);
    // the level offsets come back with the status: one synchronisation for both
    scan_exclusive_u32(c, level_hist, lvl_off, LEVELS + 1, part, nullptr);
    if (cudaMemcpyAsync(c.h_levels, lvl_off, sizeof(uint32_t) * (LEVELS + 1), cudaMemcpyDeviceToHost, c.stream) !=
        cudaSuccess)
        return cuda_status(c, cudaGetLastError());
    if ((st = read_status(c))) return st;
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

    // ---- compact level tables (host side, from the level offsets), built in
    // pinned staging and sent with one copy: level of each compact level
    // (u16 [LEVELS]), first compact level of a stream (u16 [256]), levels of a
    // stream (u8 [256]), compact id of a level (u8 [LEVELS], at most 256 levels)
    constexpr size_t ST_LOC = 0, ST_CBASE = ST_LOC + 2 * LEVELS, ST_NDEP = ST_CBASE + 2 * 256,
                     ST_CMAP = ST_NDEP + 256, ST_END = ST_CMAP + LEVELS;
    static_assert(ST_END <= STAGE_BYTES, "staging too small");
    const uint32_t *off = c.h_levels;
    uint16_t *level_of_compact = reinterpret_cast<uint16_t *>(c.h_stage + ST_LOC);
    uint16_t *cbase = reinterpret_cast<uint16_t *>(c.h_stage + ST_CBASE);
    uint8_t *ndep = c.h_stage + ST_NDEP;
    uint8_t *cmap = c.h_stage + ST_CMAP;
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

    uint64_t *rk0 = a.take<uint64_t>(R), *rk1 = a.take<uint64_t>(R);
    uint32_t *rv0 = a.take<uint32_t>(R), *rv1 = a.take<uint32_t>(R);
    uint32_t *hist = a.take<uint32_t>(radix_hist_elems(R));
    int64_t *ls = a.take<int64_t>(R), *le = a.take<int64_t>(R);
    uint32_t *li = a.take<uint32_t>(R);
    unsigned char *d_stage = a.take<unsigned char>(ST_END);
    const uint16_t *d_loc = reinterpret_cast<const uint16_t *>(d_stage + ST_LOC);
    const uint16_t *d_cbase = reinterpret_cast<const uint16_t *>(d_stage + ST_CBASE);
    const uint8_t *d_ndep = d_stage + ST_NDEP;
    const uint8_t *d_cmap = d_stage + ST_CMAP;
    uint32_t *deferred = a.take<uint32_t>(nt);
    unsigned *ndeferred = a.take<unsigned>(1);
    if (!deferred || !ndeferred) return OPATTR_E_OOM;
    int32_t *P = a.take<int32_t>((nt + 1) * (int64_t)(nl > 0 ? nl : 1));
    if (!rk0 || !rk1 || !rv0 || !rv1 || !hist || !ls || !le || !li || !d_stage || !P) return OPATTR_E_OOM;
    cudaMemcpyAsync(d_stage, c.h_stage, ST_END, cudaMemcpyHostToDevice, c.stream);

    // ---- kernel time order
    uint32_t *korder = nullptr;
    if (!k_sorted && K > 0) {
        korder = kernel_time_order(c, a, kern->stream, kern->start_ns, K);
        if (!korder) return OPATTR_E_OOM;
    }

    // ---- level lists, their validation, the windows and the enclosure, without
    // a synchronisation in between: a failed validation is reported at the end
    // (the enclosure reads only positions found by searches inside the level
    // lists, so non-laminar ranges give wrong answers but no stray access).
    // If ranges with equal starts were not in (start, end, index) order within
    // a level, the whole pass runs again on fully sorted ranges.
    const unsigned g = grid_for(R, 256, 65535);
    for (int attempt = 0; attempt < 2; ++attempt) {
        const bool full_sort = !r_sorted || attempt > 0;
        uint32_t *perm = nullptr;         // range indices in the order of the level sort
        if (full_sort) {
            // (start, end, index) order: sort by end, then stably by start
            uint64_t *ko;
            uint32_t *vo;
            int bits = bits_for((uint64_t)(rmax - rmin));
            launch(c, "range_time_key", k_time_key, dim3(g), dim3(256), 0, rng->end_ns, (const uint32_t *)nullptr, R,
                   rmin, rk0);
            radix_sort_pairs<uint64_t>(c, rk0, rv0, rk1, rv1, R, bits, true, hist, part, &ko, &vo);
            uint64_t *kfree = ko == rk0 ? rk1 : rk0;
            uint32_t *vfree = vo == rv0 ? rv1 : rv0;
            launch(c, "range_time_key", k_time_key, dim3(g), dim3(256), 0, rng->start_ns, (const uint32_t *)vo, R,
                   rmin, kfree);
            radix_sort_pairs<uint64_t>(c, kfree, vo, ko, vfree, R, bits, false, hist, part, &ko, &perm);
        }
        if (nl <= 256) {
            // stable partition by compact level id, ranges written in place
            const LevelDigit dg{rng->stream, rng->depth, d_cmap, perm};
            digit_offsets(c, dg, R, hist, part);
            const int64_t ntiles = (R + RADIX_TILE - 1) / RADIX_TILE;
            launch(c, "level_place", k_level_place, dim3((unsigned)ntiles), dim3(RADIX_THREADS), 0, dg,
                   rng->start_ns, rng->end_ns, rng->op_id, R, (const uint32_t *)hist, ntiles, ls, le, li);
        } else {
            // stable partition by level key (13 bits)
            uint32_t *lk0 = reinterpret_cast<uint32_t *>(rk0), *lk1 = reinterpret_cast<uint32_t *>(rk1);
            uint32_t *va = perm ? perm : rv0;
            uint32_t *vb = perm == rv0 ? rv1 : (perm == rv1 ? rv0 : rv1);
            launch(c, "level_keys", k_level_keys, dim3(g), dim3(256), 0, rng->stream, rng->depth,
                   (const uint32_t *)perm, R, lk0);
            uint32_t *ko32, *lperm;
            radix_sort_pairs<uint32_t>(c, lk0, va, lk1, vb, R, 13, perm == nullptr, hist, part, &ko32, &lperm);
            launch(c, "level_gather", k_level_gather, dim3(g), dim3(256), 0, rng->start_ns, rng->end_ns, rng->op_id,
                   (const uint32_t *)lperm, R, ls, le, li);
        }
        launch(c, "validate_levels", k_validate_levels, dim3(grid_for(R, 256, 65535)), dim3(256), 0, rng->stream,
               rng->depth, (const int64_t *)ls, (const int64_t *)le, (const uint32_t *)li, (const uint32_t *)lvl_off,
               R, c.d_status);
        if (K > 0 && nl == 0)
            launch(c, "fill_unattributed", k_fill_unattributed, dim3(grid_for(K, 256, 65535)), dim3(256), 0, out_range,
                   out_nop, K);
        if (K > 0 && nl > 0) {
            // chunks of WT_CHUNK tiles once the table is large (searches for
            // every entry in parallel would then repeat most of their steps)
            const int wt_chunk = (nt + 1) * (int64_t)nl >= ((int64_t)1 << 22) ? WT_CHUNK : 1;
            launch(c, "window_table", k_window_table,
                   dim3(grid_for((nt + 1 + wt_chunk - 1) / wt_chunk * nl, 256, 65535)), dim3(256), 0,
                   (const int64_t *)ls, (const uint32_t *)lvl_off, (const uint16_t *)d_loc, nl, kern->start_ns,
                   (const uint32_t *)korder, K, nt, wt_chunk, P);
            EncArgs A;
            A.k_stream = kern->stream;
            A.k_start = kern->start_ns;
            A.korder = korder;
            A.K = K;
            A.ls = ls;
            A.le = le;
            A.li = li;
            A.lvl_off = lvl_off;
            A.P = P;
            A.nl = nl;
            A.nt = nt;
            A.cbase = d_cbase;
            A.level_of_compact = d_loc;
            A.ndepth = d_ndep;
            A.out_range = out_range;
            A.out_nop = out_nop;
            static unsigned attr_done = 0;
            if (c.device < 32 && !(attr_done & (1u << c.device))) {
                cudaFuncSetAttribute(k_enclose, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(EncSmemSmall));
                cudaFuncSetAttribute(k_enclose_wide, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)sizeof(EncSmemWide));
                attr_done |= 1u << c.device;
            }
            A.tiles = nullptr;
            A.ntiles = nullptr;
            A.deferred = deferred;
            A.ndeferred = ndeferred;
            if (nl <= ENC_ACT_SMALL) {
                // compact layout first; the tiles it defers go through the wide one
                cudaMemsetAsync(ndeferred, 0, sizeof(unsigned), c.stream);
                launch(c, "enclose", k_enclose, dim3((unsigned)nt), dim3(ENC_THREADS), sizeof(EncSmemSmall), A);
                A.tiles = deferred;
                A.ntiles = ndeferred;
                int sms = 0;
                cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
                launch(c, "enclose_wide", k_enclose_wide, dim3((unsigned)std::min<int64_t>(nt, 3 * std::max(1, sms))),
                       dim3(ENC_THREADS), sizeof(EncSmemWide), A);
            } else {
                launch(c, "enclose_wide", k_enclose_wide, dim3((unsigned)nt), dim3(ENC_THREADS), sizeof(EncSmemWide),
                       A);
            }
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
        if (c.h_status->flags & F_LEVEL_FIXUP) return OPATTR_E_CUDA;   // a full sort leaves no such disorder
        return OPATTR_OK;
    }
    return OPATTR_E_CUDA;
}

}  // namespace opattr
