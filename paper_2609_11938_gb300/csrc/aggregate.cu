// aggregate.cu -- per-operator aggregation, Eq. (1) and Sec. 3.8.1, with the
// rule of each counter from Table 8, and the attributed / unattributed
// totals of Fig. 3.
//
// Fast path (kernels in time order, ranges in start order, one range per op
// id).  The kernels are cut into tiles of AGG_TILE in time order.  A range is
// owned by the tile whose time span contains its start; every kernel a range
// encloses starts at or after that, so the owner sees all of them: those in
// its own tile through a stable in-tile sort by owner slot, and the rest by
// scanning forward past the tile until the range has ended.  One thread per
// owned range accumulates its kernels in index order and writes the op's
// record once -- no atomics on op records, no partial records.  Op ids no
// range refers to are filled afterwards from a bitmap.  A kernel count check
// guards the path; if it fails (range_of_kernel inconsistent with the
// timestamps), the general path runs.
//
// General path.  Attributed kernels, in index order, are stably radix-sorted
// by op id; one thread per op id walks its segment.
//
// Accumulation is float-float with exact int64 weights (ff.cuh).
#include <stdlib.h>
#include <string.h>

#include <algorithm>

#include "ff.cuh"
#include "sort.cuh"
#include "util.cuh"

namespace opattr {

constexpr int NC = OPATTR_N_COUNTERS;
// Table 8, counter #k at index k-1: SUM #1 #2 #3 #11 #15 #19, MAX #18 #20,
// duration-weighted mean for the other twelve.
constexpr int N_SUM = 6, N_DW = 12, N_MAX = 2;

struct AggIn {
    const int64_t *dur;
    const int32_t *ncu_idx;
    const float *counters;
    int64_t n_ops;
    opattr_op_aggregates out;
};

// One operator's running aggregate.
//  kc, dsum       attributed kernels and their summed duration
//  mc, dall       matched kernels (with a row) and their summed duration
//  s[i]           SUM counters, float-float
//  w[i], nanw[i]  DW counters: sum of m*d, float-float, and the duration of
//                 matched kernels whose value was null (weight = dall - nanw)
//  mx[i]          MAX counters
constexpr int RENORM = 128;

// Per-counter finishing steps, kept out of line: they run once per operator
// and counter, and one copy keeps the kernel's instruction footprint small.
__device__ __noinline__ double finish_sum(float hi, float lo) {
    ff v{hi, lo};
    ff_renorm(v);
    return ff_to_f64(v);
}
__device__ __noinline__ double finish_dw(float hi, float lo, long long den) {
    ff v{hi, lo};
    ff_renorm(v);
    return ff_div_i64_to_f64(v, den);
}
__device__ __noinline__ double finish_max(float x) { return f32_to_f64_bits(x); }
constexpr unsigned ALL_COUNTERS = (1u << NC) - 1;

struct Acc {
    int kc, mc;
    long long dsum, dall;
    ff s[N_SUM];
    ff w[N_DW];
    long long nanw[N_DW];
    float mx[N_MAX];
    unsigned seen;      // bit c: counter c had a non-null value
    int bad;            // an infinite counter was seen
    int terms;          // accumulations since the last renormalisation

    __device__ __forceinline__ void init() {
        kc = mc = 0;
        dsum = dall = 0;
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) s[i] = ff{0.f, 0.f};
#pragma unroll
        for (int i = 0; i < N_DW; ++i) { w[i] = ff{0.f, 0.f}; nanw[i] = 0; }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) mx[i] = -INFINITY;
        seen = 0;
        bad = 0;
        terms = 0;
    }

    __device__ __forceinline__ static int sum_col(int i) {
        return i == 0 ? 0 : i == 1 ? 1 : i == 2 ? 2 : i == 3 ? 10 : i == 4 ? 14 : 18;
    }
    __device__ __forceinline__ static int dw_col(int i) { return i < 7 ? 3 + i : (i < 10 ? 4 + i : 5 + i); }
    __device__ __forceinline__ static int max_col(int i) { return i == 0 ? 17 : 19; }

    // Adds one kernel: duration d, and its counter row when `matched`.
    __device__ __forceinline__ void accumulate(long long d, bool matched, const float4 *row) {
        kc++;
        dsum += d;
        if (!matched) return;
        mc++;
        dall += d;
        float v[NC];
#pragma unroll
        for (int q = 0; q < NC / 4; ++q) {
            const float4 x = row[q];
            v[4 * q] = x.x; v[4 * q + 1] = x.y; v[4 * q + 2] = x.z; v[4 * q + 3] = x.w;
        }
        float z = 0.f;              // NaN iff some value is NaN or infinite
#pragma unroll
        for (int c = 0; c < NC; ++c) z = __fmaf_rn(v[c], 0.f, z);
        unsigned valid = ALL_COUNTERS;
        if (z != z) {
            // rare: null (NaN) values take no part -- a zero value with a
            // zero weight for the sums, -inf for the maxima -- and their
            // durations leave the DW weights; infinite values are errors
#pragma unroll
            for (int c = 0; c < NC; ++c) {
                if (isnan(v[c])) {
                    valid &= ~(1u << c);
                    v[c] = (c == 17 || c == 19) ? -INFINITY : 0.f;
                } else if (isinf(v[c])) {
                    bad = 1;
                    valid &= ~(1u << c);
                    v[c] = (c == 17 || c == 19) ? -INFINITY : 0.f;
                }
            }
#pragma unroll
            for (int i = 0; i < N_DW; ++i)
                if (!((valid >> dw_col(i)) & 1u)) nanw[i] += d;
        }
        seen |= valid;
        const ff dd = split_i64(d);
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) ff_accum(s[i], v[sum_col(i)], 0.f);
#pragma unroll
        for (int i = 0; i < N_DW; ++i) {
            const ff p = mul_split(v[dw_col(i)], dd);
            ff_accum(w[i], p.hi, p.lo);
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) mx[i] = fmaxf(mx[i], v[max_col(i)]);
        if (++terms >= RENORM) {
            terms = 0;
#pragma unroll
            for (int i = 0; i < N_SUM; ++i) ff_renorm(s[i]);
#pragma unroll
            for (int i = 0; i < N_DW; ++i) ff_renorm(w[i]);
        }
    }

    __device__ __forceinline__ void write(const AggIn &A, int64_t op) const {
        A.out.kernel_count[op] = kc;
        A.out.total_duration_ns[op] = dsum;
        A.out.matched_count[op] = mc;
        double *agg = A.out.agg;
        const int64_t n = A.n_ops;
        const double qnan = __longlong_as_double(0x7FF8000000000000ll);
#pragma unroll
        for (int i = 0; i < N_SUM; ++i)
            agg[(int64_t)sum_col(i) * n + op] = ((seen >> sum_col(i)) & 1u) ? finish_sum(s[i].hi, s[i].lo) : qnan;
#pragma unroll
        for (int i = 0; i < N_DW; ++i) {
            const long long den = dall - nanw[i];
            agg[(int64_t)dw_col(i) * n + op] =
                (((seen >> dw_col(i)) & 1u) && den > 0) ? finish_dw(w[i].hi, w[i].lo, den) : qnan;
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i)
            agg[(int64_t)max_col(i) * n + op] = ((seen >> max_col(i)) & 1u) ? finish_max(mx[i]) : qnan;
    }

    // Row fetched from global memory (general path).
    __device__ __forceinline__ void add(const AggIn &A, int64_t k) {
        const long long d = A.dur[k];
        const int32_t j = A.ncu_idx[k];
        accumulate(d, j >= 0, reinterpret_cast<const float4 *>(A.counters + (int64_t)(j >= 0 ? j : 0) * NC));
    }
};

// ------------------------------------------------------------------ checks and totals
// Per kernel: duration >= 0, range index in [-1, R), an attributed range is an
// operator below n_ops, row index in [-1, M).  Totals: all / attributed time,
// attributed and matched kernel counts.
__global__ void k_agg_check_kernels(const int64_t *__restrict__ dur, const int32_t *__restrict__ rok,
                                    const int32_t *__restrict__ nidx, const uint32_t *__restrict__ r_op, int64_t K,
                                    int64_t R, int64_t M, int64_t n_ops, DevStatus *st) {
    constexpr int U = 4;                    // kernels per thread per round, loads issued together
    unsigned long long tot = 0, att = 0, natt = 0, nmatch = 0;
    int bad = 0, not_id = 0;
    for (int64_t base = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * U; base < K;
         base += (int64_t)gridDim.x * blockDim.x * U) {
        long long d[U];
        int32_t r[U], j[U];
        uint32_t op[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const bool in = base + u < K;
            d[u] = in ? dur[base + u] : 0;
            r[u] = in ? rok[base + u] : -1;
            j[u] = in ? nidx[base + u] : -1;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) op[u] = (r[u] >= 0 && r[u] < R) ? r_op[r[u]] : 0u;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (base + u >= K) continue;
            not_id |= j[u] >= 0 && j[u] != base + u;
            if (d[u] < 0 || r[u] < -1 || r[u] >= R || j[u] < -1 || j[u] >= M) { bad = 1; continue; }
            tot += (unsigned long long)d[u];
            if (r[u] >= 0) {
                if ((int64_t)op[u] >= n_ops) { bad = 1; continue; }
                att += (unsigned long long)d[u];
                natt++;
                nmatch += j[u] >= 0;
            }
        }
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
    if (__any_sync(0xffffffffu, not_id) && lane_id() == 0) set_flag(st, F_IDX_NOT_ID);
    block_add_u64(tot, &st->cnt[C_TOTAL_NS], red);
    block_add_u64(att, &st->cnt[C_ATTR_NS], red);
    block_add_u64(natt, &st->cnt[C_ATTR_K], red);
    block_add_u64(nmatch, &st->cnt[C_MATCHED_K], red);
}

// Per range: start order of the array; a bitmap of op ids held by operator
// ranges, flagging an id held twice.
__global__ void k_agg_check_ranges(const int64_t *__restrict__ r_start, const uint32_t *__restrict__ r_op, int64_t R,
                                   int64_t n_ops, unsigned *__restrict__ bitmap, DevStatus *st) {
    int unsorted = 0, dup = 0;
    for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
        if (r + 1 < R && r_start[r + 1] < r_start[r]) unsorted = 1;
        uint32_t op = r_op[r];
        if ((int64_t)op < n_ops) {
            unsigned bit = 1u << (op & 31);
            unsigned old = atomicOr(&bitmap[op >> 5], bit);
            if (old & bit) dup = 1;
        }
    }
    if (__any_sync(0xffffffffu, unsorted) && lane_id() == 0) set_flag(st, F_R_UNSORTED);
    if (__any_sync(0xffffffffu, dup) && lane_id() == 0) set_flag(st, F_OP_DUP);
}

// ------------------------------------------------------------------ fast path
constexpr int AO_THREADS = 256;
constexpr int AO_WARPS = AO_THREADS / 32;
constexpr int AO_TILE = 1024;                    // kernels per tile
constexpr int AO_PER_WARP = AO_TILE / AO_WARPS;  // 128
constexpr int AO_OPEN = 192;                     // open ranges carried from tile to tile
constexpr int AO_KEYS = 640;                     // group keys per pass: owned slots, then carried slots
constexpr int AO_OWN = AO_KEYS - AO_OPEN;        // owned ranges per pass
constexpr int AO_HASH = 512;                     // range id -> carried slot, open addressing
constexpr unsigned AO_NONE = GROUP_NONE;
constexpr int AO_LBUCKETS = 64;

// band[t] = number of ranges with start <= T(t * AO_TILE - 1), band[0] = 0,
// band[nt] = R: tile t owns ranges [band[t], band[t+1]).
__global__ void k_band_table(const int64_t *__restrict__ k_start, int64_t K, const int64_t *__restrict__ r_start,
                             int64_t R, int64_t nt, int64_t *__restrict__ band) {
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t <= nt; t += (int64_t)gridDim.x * blockDim.x) {
        if (t == 0) { band[0] = 0; continue; }
        if (t == nt) { band[nt] = R; continue; }
        long long b = k_start[t * AO_TILE - 1];
        int64_t lo = 0, hi = R;
        while (lo < hi) {
            int64_t m = (lo + hi) >> 1;
            if (r_start[m] <= b) lo = m + 1; else hi = m;
        }
        band[t] = lo;
    }
}

struct OwnArgs {
    AggIn in;
    int64_t M;
    int identity;               // ncu_idx[k] is k or -1 for every kernel
    const int64_t *k_start;
    const int32_t *rok;
    int64_t K;
    const int64_t *r_end;
    const uint32_t *r_op;
    const int64_t *band;
    int64_t nt, tiles_per_block;
    long long wait_cycles;      // bound on the wait for a tile's bulk copy
    int withhold_copy;          // fault injection: announce the first copy but never issue it
    Acc *open_acc;              // [gridDim.x][2][AO_OPEN] carried accumulators (L2-resident scratch)
    int32_t *open_range;        // [gridDim.x][2][AO_OPEN]
    DevStatus *st;
};

struct OwnSmem {
    float4 rows[AO_TILE * (NC / 4)];   // the tile's counter rows (bulk copy or gather)
    int32_t rok[AO_TILE];
    uint16_t klist[AO_TILE];
    uint16_t wcnt[AO_WARPS][AO_KEYS];
    uint16_t soff[AO_KEYS + 1];
    uint16_t order[AO_KEYS];
    uint32_t lcount[AO_LBUCKETS + 1];
    int32_t hkey[AO_HASH];
    int16_t hval[AO_HASH];
    unsigned long long mbar;
    uint32_t wbuf[33];
    unsigned long long red[33];
    long long max_end_in, max_end_out;
    int nopen_in, nopen_out, ok;
};

// ---- bulk copy (TMA) helpers: one mbarrier per block, one copy per tile
__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(unsigned long long *bar) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void bulk_copy_g2s(void *dst, const void *src, unsigned bytes, unsigned long long *bar) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     smem_u32(dst)),
                 "l"(src), "r"(bytes), "r"(smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ bool mbar_test_wait(unsigned long long *bar, unsigned parity) {
    unsigned ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait (non-blocking polls): gives up after `limit` cycles.
__device__ __forceinline__ bool mbar_wait(unsigned long long *bar, unsigned parity, long long limit) {
    const long long t0 = clock64();
    while (!mbar_test_wait(bar, parity))
        if (clock64() - t0 > limit) return false;
    return true;
}

template <typename KeyFn>
__device__ __forceinline__ void group_by_key(OwnSmem &S, int nkeys, KeyFn key_of) {
    block_group_by_key<AO_THREADS, AO_PER_WARP>(nkeys, key_of, &S.wcnt[0][0], AO_KEYS, S.soff, S.klist, S.wbuf);
}

__device__ __forceinline__ unsigned hash_slot(int32_t r) { return ((uint32_t)r * 2654435761u) >> 23; }   // 9 bits

__device__ __forceinline__ int hash_find(const OwnSmem &S, int32_t r) {
    unsigned h = hash_slot(r);
    for (int probe = 0; probe < AO_HASH; ++probe) {
        const int32_t k = S.hkey[h];
        if (k == r) return S.hval[h];
        if (k < 0) return -1;
        h = (h + 1) & (AO_HASH - 1);
    }
    return -1;
}

// Persistent blocks: block b takes tiles [b * tpb, (b + 1) * tpb) in order.
// A range still open at the end of a tile keeps its accumulator in the
// block's carry table and picks up its kernels in the next tile.  After its
// own tiles, the block keeps walking the following tiles -- owning nothing
// there -- until every range it carries has ended.  Each tile's counter rows
// arrive in shared memory with one bulk copy (identity row map) or a gather.
__global__ void __launch_bounds__(AO_THREADS, 2) k_agg_owned(OwnArgs A) {
    extern __shared__ __align__(128) unsigned char smem_raw[];
    OwnSmem &S = *reinterpret_cast<OwnSmem *>(smem_raw);
    const int64_t t_begin = (int64_t)blockIdx.x * A.tiles_per_block;
    const int64_t t_end = t_begin + A.tiles_per_block < A.nt ? t_begin + A.tiles_per_block : A.nt;
    Acc *acc_tab[2] = {A.open_acc + (size_t)blockIdx.x * 2 * AO_OPEN, A.open_acc + ((size_t)blockIdx.x * 2 + 1) * AO_OPEN};
    int32_t *rng_tab[2] = {A.open_range + (size_t)blockIdx.x * 2 * AO_OPEN,
                           A.open_range + ((size_t)blockIdx.x * 2 + 1) * AO_OPEN};
    int cur = 0;
    unsigned phase = 0;
    unsigned long long seen = 0;
    int bad = 0;
    if (threadIdx.x == 0) {
        mbar_init(&S.mbar);
        S.nopen_in = 0;
        S.max_end_in = LLONG_MIN;
    }
    __syncthreads();

    for (int64_t t = t_begin; t < A.nt; ++t) {
        const bool own = t < t_end;
        if (!own && (S.nopen_in == 0 || A.k_start[t * AO_TILE] > S.max_end_in)) break;
        const int64_t k0 = t * AO_TILE;
        const int64_t kn = A.K - k0 < AO_TILE ? A.K - k0 : AO_TILE;
        const int64_t k1 = k0 + kn;
        const int64_t ra = own ? A.band[t] : 0, rb = own ? A.band[t + 1] : 0;
        const long long t_next = k1 < A.K ? A.k_start[k1] : LLONG_MAX;
        const int nin = S.nopen_in;
        // ---- stage the tile: rows (bulk copy or gather), range ids, carried-range hash
        int64_t nrows = A.identity ? (A.M - k0 < kn ? A.M - k0 : kn) : 0;
        if (nrows < 0) nrows = 0;
        if (threadIdx.x == 0 && nrows > 0) {
            if (A.withhold_copy && t == t_begin)
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(&S.mbar)),
                             "r"((unsigned)(nrows * NC * 4))
                             : "memory");
            else
                bulk_copy_g2s(S.rows, A.in.counters + k0 * NC, (unsigned)(nrows * NC * 4), &S.mbar);
        }
        for (int i = threadIdx.x; i < AO_TILE; i += AO_THREADS) S.rok[i] = i < kn ? A.rok[k0 + i] : -1;
        if (!A.identity) {
            for (int i = threadIdx.x; i < kn; i += AO_THREADS) {
                const int32_t j = A.in.ncu_idx[k0 + i];
                if (j < 0) continue;
                const float4 *src = reinterpret_cast<const float4 *>(A.in.counters + (int64_t)j * NC);
#pragma unroll
                for (int q = 0; q < NC / 4; ++q) S.rows[i * (NC / 4) + q] = __ldg(src + q);
            }
        }
        for (int i = threadIdx.x; i < AO_HASH; i += AO_THREADS) S.hkey[i] = -1;
        if (threadIdx.x == 0) { S.nopen_out = 0; S.max_end_out = LLONG_MIN; S.ok = 1; }
        __syncthreads();
        for (int o = threadIdx.x; o < nin; o += AO_THREADS) {
            const int32_t r = rng_tab[cur][o];
            unsigned h = hash_slot(r);
            for (int probe = 0; probe < AO_HASH && atomicCAS(&S.hkey[h], -1, r) != -1; ++probe)
                h = (h + 1) & (AO_HASH - 1);
            S.hval[h] = (int16_t)o;
        }
        if (threadIdx.x == 0 && nrows > 0) {
            if (!mbar_wait(&S.mbar, phase, A.wait_cycles)) {
                // give up on this launch, but let the copy land before the block exits
                set_err(A.st, ERR_TIMEOUT);
                mbar_wait(&S.mbar, phase, 64 * A.wait_cycles + (1ll << 24));
                S.ok = 0;
            }
        }
        if (nrows > 0) phase ^= 1u;
        __syncthreads();
        if (!S.ok) return;
        // ---- passes over the owned ranges; the carried ranges join the first
        bool first = true;
        for (int64_t ca = ra; first || ca < rb; ca += AO_OWN, first = false) {
            const int64_t cb = rb - ca < AO_OWN ? rb : ca + AO_OWN;
            const int nown = cb > ca ? (int)(cb - ca) : 0;
            const int ncar = first ? nin : 0;
            if (nown == 0 && ncar == 0) break;
            group_by_key(S, nown + ncar, [&](int i) -> unsigned {
                const int32_t r = S.rok[i];
                if (r < 0) return (unsigned)AO_NONE;
                if (r >= ca && r < cb) return (unsigned)(r - ca);
                if (ncar) {
                    const int o = hash_find(S, r);
                    if (o >= 0) return (unsigned)(nown + o);
                }
                return (unsigned)AO_NONE;
            });
            // ranges ordered by kernel count, longest first (counting sort on
            // a capped length), dealt out snake-wise for balance
            const int nact = nown + ncar;
            for (int i = threadIdx.x; i <= AO_LBUCKETS; i += AO_THREADS) S.lcount[i] = 0;
            __syncthreads();
            for (int a = threadIdx.x; a < nact; a += AO_THREADS) {
                const int len = S.soff[a + 1] - S.soff[a];
                atomicAdd(&S.lcount[AO_LBUCKETS - 1 - (len < AO_LBUCKETS - 1 ? len : AO_LBUCKETS - 1)], 1u);
            }
            __syncthreads();
            if (threadIdx.x == 0) {
                unsigned run = 0;
                for (int b = 0; b < AO_LBUCKETS; ++b) { unsigned x = S.lcount[b]; S.lcount[b] = run; run += x; }
            }
            __syncthreads();
            for (int a = threadIdx.x; a < nact; a += AO_THREADS) {
                const int len = S.soff[a + 1] - S.soff[a];
                const unsigned pos = atomicAdd(&S.lcount[AO_LBUCKETS - 1 - (len < AO_LBUCKETS - 1 ? len : AO_LBUCKETS - 1)], 1u);
                S.order[pos] = (uint16_t)a;
            }
            __syncthreads();
            for (int g = 0; g * AO_THREADS < nact; ++g) {
                const int a = g * AO_THREADS + ((g & 1) ? AO_THREADS - 1 - (int)threadIdx.x : (int)threadIdx.x);
                if (a >= nact) continue;
                const int key = S.order[a];
                int64_t r;
                Acc acc;
                if (key < nown) {
                    r = ca + key;
                    if ((int64_t)A.r_op[r] >= A.in.n_ops) continue;   // not an operator range
                    acc.init();
                } else {
                    const int o = key - nown;
                    r = rng_tab[cur][o];
                    acc = acc_tab[cur][o];
                }
                for (int q = S.soff[key]; q < S.soff[key + 1]; ++q) {
                    const int i = S.klist[q];
                    const int64_t k = k0 + i;
                    acc.accumulate(A.in.dur[k], A.in.ncu_idx[k] >= 0, &S.rows[i * (NC / 4)]);
                }
                const long long e = A.r_end[r];
                if (e >= t_next) {
                    const int o2 = atomicAdd(&S.nopen_out, 1);
                    if (o2 < AO_OPEN) {
                        acc_tab[cur ^ 1][o2] = acc;
                        rng_tab[cur ^ 1][o2] = (int32_t)r;
                        atomicMax(&S.max_end_out, e);
                    } else {
                        set_flag(A.st, F_AGG_MISS);             // carry table full: the general path redoes it
                    }
                    continue;
                }
                acc.write(A.in, A.r_op[r]);
                seen += (unsigned long long)acc.kc;
                bad |= acc.bad;
            }
            __syncthreads();
        }
        if (threadIdx.x == 0) {
            S.nopen_in = S.nopen_out < AO_OPEN ? S.nopen_out : AO_OPEN;
            S.max_end_in = S.max_end_out;
        }
        cur ^= 1;
        __syncthreads();
    }
    // ranges still carried here ended before the next tile
    for (int o = threadIdx.x; o < S.nopen_in; o += AO_THREADS) {
        const Acc acc = acc_tab[cur][o];
        acc.write(A.in, A.r_op[rng_tab[cur][o]]);
        seen += (unsigned long long)acc.kc;
        bad |= acc.bad;
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(A.st, ERR_INVALID);
    block_add_u64(seen, &A.st->cnt[C_AGG_SEEN], S.red);
}

// Op ids held by no operator range: empty records.
__global__ void k_agg_fill_unreferenced(const unsigned *__restrict__ bitmap, AggIn A) {
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < A.n_ops; o += (int64_t)gridDim.x * blockDim.x) {
        if ((bitmap[o >> 5] >> (o & 31)) & 1u) continue;
        Acc acc;
        acc.init();
        acc.write(A, o);
    }
}

// ------------------------------------------------------------------ general path
__global__ void k_agg_attr_flags(const int32_t *__restrict__ rok, int64_t K, uint32_t *__restrict__ flag) {
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x)
        flag[k] = rok[k] >= 0;
}
__global__ void k_agg_attr_keys(const int32_t *__restrict__ rok, const uint32_t *__restrict__ r_op,
                                const uint32_t *__restrict__ flag, const uint32_t *__restrict__ pos, int64_t K,
                                uint32_t *__restrict__ keys, uint32_t *__restrict__ kidx) {
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x)
        if (flag[k]) {
            keys[pos[k]] = r_op[rok[k]];
            kidx[pos[k]] = (uint32_t)k;
        }
}
__global__ void k_agg_general(const uint32_t *__restrict__ sop, const uint32_t *__restrict__ sj,
                              const uint32_t *__restrict__ kidx, int64_t n, AggIn A, DevStatus *st) {
    int bad = 0;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < A.n_ops; o += (int64_t)gridDim.x * blockDim.x) {
        int64_t lo = 0, hi = n;
        while (lo < hi) {
            int64_t m = (lo + hi) >> 1;
            if (sop[m] < (uint32_t)o) lo = m + 1; else hi = m;
        }
        Acc acc;
        acc.init();
        for (int64_t i = lo; i < n && sop[i] == (uint32_t)o; ++i) acc.add(A, kidx[sj[i]]);
        acc.write(A, o);
        bad |= acc.bad;
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
}

// ------------------------------------------------------------------ host
opattr_status do_aggregate(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                           const opattr_ncu *ncu, const int32_t *nidx, uint32_t n_ops,
                           const opattr_op_aggregates *out, opattr_totals *tot_out) {
    const int64_t K = kern->n, R = rng->n, M = ncu->n, O = n_ops;
    if (K < 0 || R < 0 || M < 0 || K >= (1ll << 31) || R >= (1ll << 31) || M >= (1ll << 31) || !out)
        return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->dur_ns || !rok || !nidx || (!kern->start_ns) || (!kern->stream))) return OPATTR_E_INVALID_ARG;
    if (R > 0 && (!rng->op_id || !rng->start_ns || !rng->end_ns)) return OPATTR_E_INVALID_ARG;
    if (M > 0 && !ncu->counters) return OPATTR_E_INVALID_ARG;
    if (O > 0 && (!out->kernel_count || !out->total_duration_ns || !out->matched_count || !out->agg))
        return OPATTR_E_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ncu->counters) & 15) != 0) return OPATTR_E_INVALID_ARG;

    const int64_t nt = (K + AO_TILE - 1) / AO_TILE;   // tiles of the owned-range path
    int sms = 0, per_sm = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
    {
        static unsigned attr_done = 0;
        if (c.device < 32 && !(attr_done & (1u << c.device))) {
            cudaFuncSetAttribute(k_agg_owned, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sizeof(OwnSmem));
            attr_done |= 1u << c.device;
        }
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_agg_owned, AO_THREADS, sizeof(OwnSmem));
        cudaGetLastError();
    }
    const int64_t max_grid = (int64_t)std::max(1, sms) * std::max(1, per_sm);
    const int64_t tpb = std::max<int64_t>(1, (nt + max_grid - 1) / max_grid);
    const int64_t ogrid = nt > 0 ? (nt + tpb - 1) / tpb : 1;
    Need nd;
    nd.add<unsigned>((O + 31) / 32 + 1).add<int64_t>(nt + 1);
    nd.add<Acc>(ogrid * 2 * AO_OPEN).add<int32_t>(ogrid * 2 * AO_OPEN);
    for (int i = 0; i < 7; ++i) nd.add<uint32_t>(K);
    nd.add<uint32_t>(radix_hist_elems(K)).add<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), K)));
    opattr_status st = ensure_arena(c, nd.bytes + 4096);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;
    unsigned *bitmap = a.take<unsigned>((O + 31) / 32 + 1);
    int64_t *band = a.take<int64_t>(nt + 1);
    Acc *open_acc = a.take<Acc>(ogrid * 2 * AO_OPEN);
    int32_t *open_range = a.take<int32_t>(ogrid * 2 * AO_OPEN);
    if (!bitmap || !band || !open_acc || !open_range) return OPATTR_E_OOM;
    cudaMemsetAsync(bitmap, 0, sizeof(unsigned) * ((O + 31) / 32 + 1), c.stream);
    if (K > 0) {
        launch(c, "agg_check_kernels", k_agg_check_kernels, dim3(grid_for(K, 256 * 16, REDUCE_GRID)), dim3(256), 0, kern->dur_ns,
               rok, nidx, rng->op_id, K, R, M, O, c.d_status);
        check_kernel_order(c, kern->stream, kern->start_ns, K);
    }
    if (R > 0)
        launch(c, "agg_check_ranges", k_agg_check_ranges, dim3(grid_for(R, 256 * 8, REDUCE_GRID)), dim3(256), 0, rng->start_ns,
               rng->op_id, R, O, bitmap, c.d_status);
    if ((st = read_status(c))) return st;
    if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    opattr_totals T{};
    T.total_ns = (int64_t)c.h_status->cnt[C_TOTAL_NS];
    T.attributed_ns = (int64_t)c.h_status->cnt[C_ATTR_NS];
    T.unattributed_ns = T.total_ns - T.attributed_ns;
    T.kernels = K;
    T.attributed_kernels = (int64_t)c.h_status->cnt[C_ATTR_K];
    T.matched_kernels = (int64_t)c.h_status->cnt[C_MATCHED_K];
    const double qnan = __builtin_nan("");
    T.attributed_frac = T.total_ns > 0 ? (double)T.attributed_ns / (double)T.total_ns : qnan;
    T.unattributed_frac = T.total_ns > 0 ? (double)T.unattributed_ns / (double)T.total_ns : qnan;
    if (O == 0) {
        if (tot_out) *tot_out = T;
        return OPATTR_OK;
    }
    AggIn in;
    in.dur = kern->dur_ns;
    in.ncu_idx = nidx;
    in.counters = ncu->counters;
    in.n_ops = O;
    in.out = *out;
    const unsigned flags = c.h_status->flags;
    bool fast = K > 0 && !(flags & (F_K_UNSORTED | F_R_UNSORTED | F_OP_DUP));
    if (fast) {
        launch(c, "band_table", k_band_table, dim3(grid_for(nt + 1, 256, 65535)), dim3(256), 0, kern->start_ns, K,
               rng->start_ns, R, nt, band);
        OwnArgs A;
        A.in = in;
        A.M = M;
        A.identity = !(flags & F_IDX_NOT_ID);
        A.k_start = kern->start_ns;
        A.rok = rok;
        A.K = K;
        A.r_end = rng->end_ns;
        A.r_op = rng->op_id;
        A.band = band;
        A.nt = nt;
        A.tiles_per_block = tpb;
        A.wait_cycles = c.cfg.spin_limit > 0 ? c.cfg.spin_limit : (1ll << 31);
        {
            const char *fault = getenv("OPATTR_FAULT");
            A.withhold_copy = fault && strcmp(fault, "wait") == 0;
        }
        A.open_acc = open_acc;
        A.open_range = open_range;
        A.st = c.d_status;
        launch(c, "agg_owned", k_agg_owned, dim3((unsigned)ogrid), dim3(AO_THREADS), sizeof(OwnSmem), A);
        launch(c, "agg_fill_unreferenced", k_agg_fill_unreferenced, dim3(grid_for(O, 256, 65535)), dim3(256), 0,
               (const unsigned *)bitmap, in);
        if ((st = read_status(c))) return st;
        if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
        if (c.h_status->err & ERR_TIMEOUT) return OPATTR_E_TIMEOUT;
        fast = !(c.h_status->flags & F_AGG_MISS) && c.h_status->cnt[C_AGG_SEEN] == c.h_status->cnt[C_ATTR_K];
    }
    if (!fast) {
        uint32_t *flag = a.take<uint32_t>(K), *pos = a.take<uint32_t>(K), *keys = a.take<uint32_t>(K);
        uint32_t *kidx = a.take<uint32_t>(K), *s0 = a.take<uint32_t>(K), *s1 = a.take<uint32_t>(K),
                 *s2 = a.take<uint32_t>(K);
        uint32_t *hist = a.take<uint32_t>(radix_hist_elems(K));
        uint32_t *part = a.take<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), K)));
        if (!flag || !pos || !keys || !kidx || !s0 || !s1 || !s2 || !hist || !part) return OPATTR_E_OOM;
        const int64_t natt = T.attributed_kernels;
        uint32_t *sop = keys, *sj = s0;
        if (K > 0) {
            launch(c, "agg_attr_flags", k_agg_attr_flags, dim3(grid_for(K, 256, 65535)), dim3(256), 0, rok, K, flag);
            scan_exclusive_u32(c, flag, pos, K, part, nullptr);
            launch(c, "agg_attr_keys", k_agg_attr_keys, dim3(grid_for(K, 256, 65535)), dim3(256), 0, rok, rng->op_id,
                   (const uint32_t *)flag, (const uint32_t *)pos, K, keys, kidx);
            if (natt > 0)
                radix_sort_pairs<uint32_t>(c, keys, s0, s1, s2, natt, bits_for((uint64_t)(O - 1)), true, hist, part,
                                           &sop, &sj);
        }
        launch(c, "agg_general", k_agg_general, dim3(grid_for(O, 256, 65535)), dim3(256), 0, (const uint32_t *)sop,
               (const uint32_t *)sj, (const uint32_t *)kidx, natt, in, c.d_status);
        if ((st = read_status(c))) return st;
        if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    }
    if (tot_out) *tot_out = T;
    return OPATTR_OK;
}

}  // namespace opattr
