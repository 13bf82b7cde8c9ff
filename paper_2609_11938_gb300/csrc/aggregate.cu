// aggregate.cu -- per-operator aggregation, Eq. (1) and Sec. 3.8.1, with the
// rule of each counter from Table 8, and the attributed / unattributed
// totals of Fig. 4.
//
// Operators are keyed by op id (op_id[range_of_kernel[k]]), so ranges that
// share an op id aggregate together and no order of kernels or ranges is
// needed.  Three passes over the kernels and one over the ops:
//   count  validate each kernel, add up the totals, count kernels per op id
//          and give each kernel its slot among its op's kernels
//   scan   per-op offsets into one list of attributed kernels
//   place  put each attributed kernel in its slot of its op's segment
//   ops    one thread per op id accumulates its segment in ascending kernel
//          index -- the order the count's atomics left is not used, so
//          results do not depend on it -- and writes the op's record; ops
//          without kernels get empty records in the same pass.
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
    int64_t M;                  // ncu rows: a row index at or past M is never read (the count pass reports it)
    int64_t n_ops;
    unsigned *ctr;              // [0] next chunk of the ops pass, [1] ops listed in dirty; zeroed before it
    uint32_t *dirty;            // ops whose fast sums saw a null or infinite value
    uint32_t *longs;            // ops the ops pass leaves to the pieces pass (listed there)
    unsigned *nlong;            //   and their number (zeroed before the ops pass)
    const unsigned *nonident;   // nonzero unless ncu_idx[k] == k for every kernel (set by the count pass)
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

// A duration as a normalised pair (as split_i64), the common case (< 2^48 ns)
// without branches.
__device__ __forceinline__ ff split_dur(long long d) {
    const unsigned long long u = (unsigned long long)d;
    if (u >> 48) return split_i64(d);
    const float a = __uint2float_rn((unsigned)(u >> 24)) * 16777216.0f;   // exact
    const float b = __uint2float_rn((unsigned)(u & 0xFFFFFFu));            // exact
    return fast_two_sum(a, b);                                            // |a| >= |b| or a == 0
}

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
        const bool ok = j >= 0 && j < A.M;
        accumulate(d, ok, reinterpret_cast<const float4 *>(A.counters + (int64_t)(ok ? j : 0) * NC));
    }
};

// The common case, without per-value tests: a null (NaN) or infinite value
// anywhere poisons a sum, and the op is then done again with Acc, which
// handles nulls and flags infinities.  MAX values also enter a plain sum for
// that test.  Every counter of every matched kernel is non-null here, so a
// counter is defined iff some kernel matched, and the DW weight is dall.
struct AccF {
    int mc;
    long long dsum, dall;
    ff s[N_SUM];
    ff w[N_DW];
    float mx[N_MAX];
    float probe;                // sum of the MAX values: non-finite iff one was
    int terms;

    __device__ __forceinline__ void init() {
        mc = 0;
        dsum = dall = 0;
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) s[i] = ff{0.f, 0.f};
#pragma unroll
        for (int i = 0; i < N_DW; ++i) w[i] = ff{0.f, 0.f};
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) mx[i] = -INFINITY;
        probe = 0.f;
        terms = 0;
    }

    __device__ __forceinline__ void accumulate(long long d, bool matched, const float4 *row) {
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
        const ff dd = split_dur(d);
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) {
            const ff t = two_sum(s[i].hi, v[Acc::sum_col(i)]);
            s[i].hi = t.hi;
            s[i].lo = __fadd_rn(s[i].lo, t.lo);
        }
#pragma unroll
        for (int i = 0; i < N_DW; ++i) {
            const ff p = mul_split(v[Acc::dw_col(i)], dd);
            ff_accum(w[i], p.hi, p.lo);
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) {
            mx[i] = fmaxf(mx[i], v[Acc::max_col(i)]);
            probe = __fadd_rn(probe, v[Acc::max_col(i)]);
        }
        if (++terms >= RENORM) {
            terms = 0;
#pragma unroll
            for (int i = 0; i < N_SUM; ++i) ff_renorm(s[i]);
#pragma unroll
            for (int i = 0; i < N_DW; ++i) ff_renorm(w[i]);
        }
    }

    // True when no null or infinite value took part (then write() is exact to spec).
    __device__ __forceinline__ bool clean() const {
        float z = __fmul_rn(probe, 0.f);
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) z = __fmaf_rn(__fadd_rn(s[i].hi, s[i].lo), 0.f, z);
#pragma unroll
        for (int i = 0; i < N_DW; ++i) z = __fmaf_rn(__fadd_rn(w[i].hi, w[i].lo), 0.f, z);
        return z == 0.f;
    }

    __device__ __forceinline__ void write(const AggIn &A, int64_t op, int kc) const {
        A.out.kernel_count[op] = kc;
        A.out.total_duration_ns[op] = dsum;
        A.out.matched_count[op] = mc;
        double *agg = A.out.agg;
        const int64_t n = A.n_ops;
        const double qnan = __longlong_as_double(0x7FF8000000000000ll);
        if (mc == 0) {
            // no matched kernel: every counter is null; nothing to convert
#pragma unroll
            for (int c = 0; c < NC; ++c) agg[(int64_t)c * n + op] = qnan;
            return;
        }
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) {
            ff x = s[i];
            ff_renorm(x);
            agg[(int64_t)Acc::sum_col(i) * n + op] = ff_to_f64_fast(x);
        }
        if (dall > 0) {
            const ff rcp = ff_recip_i64(dall);
#pragma unroll
            for (int i = 0; i < N_DW; ++i) agg[(int64_t)Acc::dw_col(i) * n + op] = ff_mul_to_f64(w[i], rcp);
        } else {
#pragma unroll
            for (int i = 0; i < N_DW; ++i) agg[(int64_t)Acc::dw_col(i) * n + op] = qnan;
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) agg[(int64_t)Acc::max_col(i) * n + op] = f32_to_f64_fast(mx[i]);
    }
};

// The range of kernel k; without range_of_kernel, r_op holds one operator
// per kernel and the kernel is its own "range" when it has one.
__device__ __forceinline__ int32_t range_of(const int32_t *rok, const uint32_t *r_op, int64_t k) {
    return rok ? rok[k] : (r_op[k] != OPATTR_OP_NONE ? (int32_t)k : -1);
}
template <bool DIRECT>           // DIRECT: one operator per kernel (no range_of_kernel)
__device__ __forceinline__ int32_t range_of_t(const int32_t *rok, const uint32_t *r_op, int64_t k) {
    if (DIRECT) return r_op[k] != OPATTR_OP_NONE ? (int32_t)k : -1;
    return rok[k];
}

// ------------------------------------------------------------------ count
// Per kernel: duration >= 0, range index in [-1, R), an attributed range is
// an operator below n_ops, row index in [-1, M).  Totals: all / attributed
// time, attributed and matched kernel counts.  Whether every kernel's row is
// its own index (the match of a trace whose ncu rows follow the kernels one
// for one) is noted, so the ops pass can skip the row-index gather; with
// ident_rows (a join whose matching was that identity pairing) the row
// indices are known to be the kernel indices and are not read.  Each
// attributed kernel (valid range and op id) also takes its slot among its
// op's kernels: one atomic per distinct op id of a warp on cnt[op], whose old
// value plus the kernel's rank among its warp peers is the slot (rank[k]);
// cnt ends as the per-op counts.  Each warp takes a run of `run` consecutive
// kernels (a multiple of 32, up to AF_RUN) 32 at a time in index order, so an
// op whose kernels all lie in one run gets ascending slots; the ops pass
// sorts the few segments that do not.
constexpr int AF_RUN = 4096;

template <bool DIRECT>
__global__ void __launch_bounds__(256, 5) k_agg_count(const int64_t *__restrict__ dur, const int32_t *__restrict__ rok,
                            const int32_t *__restrict__ nidx, const uint32_t *__restrict__ r_op, int64_t K, int64_t R,
                            int64_t M, int64_t n_ops, uint32_t *__restrict__ cnt, uint32_t *__restrict__ rank,
                            int64_t run, int ident_rows, unsigned *__restrict__ nonident, DevStatus *st) {
    pdl_wait();
    const unsigned lane = lane_id(), lt = lanemask_lt();
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) / 32;
    const int64_t nwarps = (int64_t)gridDim.x * blockDim.x / 32;
    unsigned long long tot = 0, att = 0, natt = 0, nmatch = 0;
    int bad = 0, nid = 0;
    auto op_of = [&](int32_t r) -> uint32_t { return (r >= 0 && r < R) ? r_op[r] : 0xFFFFFFFFu; };
    for (int64_t k0 = warp * run; k0 < K; k0 += nwarps * run) {
        const int64_t k1 = k0 + run < K ? k0 + run : K;
        // ranges two groups ahead; op ids, durations and row indices one group
        // ahead, so each step waits only on its own atomic
        int64_t k = k0 + lane;
        int32_t r_c = k < k1 ? range_of_t<DIRECT>(rok, r_op, k) : -1;
        uint32_t op_c = op_of(r_c);
        long long d_c = k < k1 ? dur[k] : 0;
        int32_t j_c = k < k1 ? (ident_rows ? (int32_t)k : nidx[k]) : -1;
        int32_t r_n = k + 32 < k1 ? range_of_t<DIRECT>(rok, r_op, k + 32) : -1;
        for (int64_t kb = k0; kb < k1; kb += 32) {
            k = kb + lane;
            const bool in = k < k1;
            const int32_t r = r_c, j = j_c;
            const uint32_t op = op_c;
            const long long d = d_c;
            r_c = r_n;
            op_c = op_of(r_n);
            d_c = k + 32 < k1 ? dur[k + 32] : 0;
            j_c = k + 32 < k1 ? (ident_rows ? (int32_t)(k + 32) : nidx[k + 32]) : -1;
            r_n = k + 64 < k1 ? range_of_t<DIRECT>(rok, r_op, k + 64) : -1;
            nid |= in && (int64_t)j != k;
            bool valid = in;
            if (in && (d < 0 || r < -1 || r >= R || j < -1 || j >= M || (r >= 0 && (int64_t)op >= n_ops))) {
                bad = 1;
                valid = false;
            }
            if (valid) {
                tot += (unsigned long long)d;
                if (r >= 0) {
                    att += (unsigned long long)d;
                    natt++;
                    nmatch += j >= 0;
                }
            }
            // slotted exactly as k_agg_place places it: by range and op id alone
            const unsigned key = (in && r >= 0 && r < R && (int64_t)op < n_ops) ? op : 0xFFFFFFFFu;
            const unsigned peers = __match_any_sync(0xffffffffu, key);
            const int leader = __ffs(peers) - 1;
            unsigned base = 0;
            if (key != 0xFFFFFFFFu && (int)lane == leader) base = atomicAdd(&cnt[key], (unsigned)__popc(peers));
            base = __shfl_sync(0xffffffffu, base, leader);
            if (key != 0xFFFFFFFFu) rank[k] = base + __popc(peers & lt);
        }
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
    if (__any_sync(0xffffffffu, nid) && lane_id() == 0) atomicOr(nonident, 1u);
    block_add_u64(tot, &st->cnt[C_TOTAL_NS], red);
    block_add_u64(att, &st->cnt[C_ATTR_NS], red);
    block_add_u64(natt, &st->cnt[C_ATTR_K], red);
    block_add_u64(nmatch, &st->cnt[C_MATCHED_K], red);
}

// ------------------------------------------------------------------ place
// list[off[op] + rank[k]] = k for each kernel k_agg_count slotted.
template <bool DIRECT>
__global__ void k_agg_place(const int32_t *__restrict__ rok, const uint32_t *__restrict__ r_op, int64_t K, int64_t R,
                            int64_t n_ops, const uint32_t *__restrict__ off, const uint32_t *__restrict__ rank,
                            uint32_t *__restrict__ list) {
    pdl_wait();
    constexpr int U = 4;                    // kernels per thread per round, loads issued together
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t k0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k0 < K; k0 += stride * U) {
        int32_t r[U];
        uint32_t op[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t k = k0 + u * stride;
            r[u] = k < K ? range_of_t<DIRECT>(rok, r_op, k) : -1;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) op[u] = (r[u] >= 0 && r[u] < R) ? r_op[r[u]] : 0xFFFFFFFFu;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t k = k0 + u * stride;
            if (r[u] >= 0 && r[u] < R && (int64_t)op[u] < n_ops) list[off[op[u]] + rank[k]] = (uint32_t)k;
        }
    }
}

// ------------------------------------------------------------------ long segments
// Segments of the ops longer than AG_HUGE (the pieces pass below) are sorted
// by kernel index first, one block per segment: up to SL_SMEM entries by a
// bitonic sort in shared memory; longer ones in SL_SMEM runs sorted that way,
// then merged pairwise through `tmp` (merge path: each thread merges an equal
// share of the output after a binary search on its diagonal).
constexpr int SL_THREADS = 256;
constexpr int SL_SMEM = 8192;

constexpr uint32_t AG_SHORT_MAX = 64;           // segments up to this length: sorted in place by one lane
constexpr uint32_t AG_HUGE = 256;               // longer segments: split into pieces over several warps
constexpr uint32_t AG_PIECE = 1024;              // kernels of a huge op per warp of the pieces pass
constexpr uint32_t AG_BLOCK_SORT_MAX = 4096;     // longer huge segments: placed by a counting pass, not sorted

__device__ void bitonic_smem(uint32_t *a, int n2) {     // n2 a power of two; the block sorts a[0..n2)
    for (int k = 2; k <= n2; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n2; i += blockDim.x) {
                const int p = i ^ j;
                if (p > i) {
                    const uint32_t x = a[i], y = a[p];
                    if (((i & k) == 0) == (x > y)) { a[i] = y; a[p] = x; }
                }
            }
            __syncthreads();
        }
}

__global__ void __launch_bounds__(SL_THREADS) k_agg_sort_long(const uint32_t *__restrict__ off,
                                                              const uint32_t *__restrict__ longs,
                                                              const unsigned *__restrict__ nlong, uint32_t min_len,
                                                              uint32_t max_len, uint32_t *list, uint32_t *tmp) {
    pdl_wait();
    __shared__ uint32_t a[SL_SMEM];
    const unsigned n_long = *nlong;
    for (unsigned li = blockIdx.x; li < n_long; li += gridDim.x) {
        const uint32_t o = longs[li], s0 = off[o], len = off[o + 1] - s0;
        if (len < min_len || len > max_len) continue;      // uniform per block
        uint32_t *seg = list + s0, *alt = tmp + s0;
        // runs of SL_SMEM (the whole segment if it fits)
        for (uint32_t r0 = 0; r0 < len; r0 += SL_SMEM) {
            const int n = (int)(len - r0 < (uint32_t)SL_SMEM ? len - r0 : (uint32_t)SL_SMEM);
            int n2 = 1;
            while (n2 < n) n2 <<= 1;
            for (int i = threadIdx.x; i < n2; i += SL_THREADS) a[i] = i < n ? seg[r0 + i] : 0xFFFFFFFFu;
            __syncthreads();
            bitonic_smem(a, n2);
            for (int i = threadIdx.x; i < n; i += SL_THREADS) seg[r0 + i] = a[i];
            __syncthreads();
        }
        // merge passes, seg -> alt -> seg ...
        uint32_t *src = seg, *dst = alt;
        for (uint32_t w = SL_SMEM; w < len; w <<= 1) {
            for (uint32_t lo = 0; lo < len; lo += 2 * w) {
                const uint32_t mid = lo + w < len ? lo + w : len, hi = lo + 2 * w < len ? lo + 2 * w : len;
                const uint32_t na = mid - lo, nb = hi - mid, total = na + nb;
                const uint32_t share = (total + SL_THREADS - 1) / SL_THREADS;
                const uint32_t d0 = threadIdx.x * share < total ? threadIdx.x * share : total;
                const uint32_t d1 = d0 + share < total ? d0 + share : total;
                // i = items taken from run a among the first d0 outputs
                uint32_t ilo = d0 > nb ? d0 - nb : 0, ihi = d0 < na ? d0 : na;
                while (ilo < ihi) {
                    const uint32_t i = (ilo + ihi) >> 1;
                    if (src[lo + i] <= src[mid + (d0 - i - 1)]) ilo = i + 1; else ihi = i;
                }
                uint32_t i = ilo, j = d0 - ilo;
                for (uint32_t d = d0; d < d1; ++d) {
                    const bool take_a = j >= nb || (i < na && src[lo + i] <= src[mid + j]);
                    dst[lo + d] = take_a ? src[lo + i++] : src[mid + j++];
                }
            }
            __syncthreads();
            uint32_t *t = src; src = dst; dst = t;
        }
        if (src != seg) {
            for (uint32_t i = threadIdx.x; i < len; i += SL_THREADS) seg[i] = src[i];
        }
        __syncthreads();
    }
}

// ------------------------------------------------------------------ ops
// One thread per op id.  Each warp takes AG_CHUNK consecutive op ids at a
// time, orders them by segment length (longest first) and walks them in
// AG_CHUNK / 32 rounds, so that the threads of a round walk segments of
// similar length and finish together (the record is written by every lane of
// the round at once); warps share nothing and never wait for each other.
// The grid is what stays resident; warps draw the chunks in increasing order
// from one counter (the next chunk is drawn, and its offsets loaded, while
// the current one runs), so the ops in flight at any moment are one narrow
// band of op ids whatever each warp's pace, and with op ids in range order
// the kernels and outputs of that band stay in L2.  The chunk's segments are
// one contiguous run of the list; when it fits it is first copied to shared
// memory by coalesced loads, and each thread checks its segments there and,
// in the rare case the count pass met an op in two runs, sorts them in place,
// so segments are walked in ascending kernel index (a larger chunk reads the
// list in place: segments up to AG_SHORT_MAX are checked and sorted there).
// Ops longer than AG_HUGE, and longer than AG_SHORT_MAX in a chunk that does
// not fit, are listed for the pieces pass instead (sorted there by a block
// each).  While a kernel is added, the counter rows and durations
// of the next two arrive in per-thread shared-memory slots by asynchronous
// copy (cp.async), with their row indices loaded a step earlier still (or
// taken to be the kernel indices when the count pass found every row to be
// its kernel's own index).
constexpr int AG_THREADS = 128;
constexpr int AG_WARPS = AG_THREADS / 32;
constexpr int AG_CHUNK = 64;                    // op ids per warp and chunk
constexpr int AG_LBUCKETS = 32;
constexpr int AG_STAGE = 1024;                  // list entries of a chunk staged in shared memory

struct OpsWarp {
    float4 row[2][32][NC / 4];      // two kernels in flight per thread: counter rows
    long long dur[2][32];           // and durations, by asynchronous copy
    uint32_t L[AG_STAGE];           // the chunk's list run (when it fits)
    uint32_t lcount[AG_LBUCKETS];
    uint8_t order[AG_CHUNK];
};
constexpr size_t AG_SMEM = sizeof(OpsWarp) * AG_WARPS;

// An op whose fast sums saw a null or infinite value: the segment again, in
// the same order, with Acc.  Returns 1 if a value was infinite.
__device__ __noinline__ int op_careful(const uint32_t *seg, uint32_t len, AggIn A, int64_t o) {
    Acc acc;
    acc.init();
    for (uint32_t t = 0; t < len; ++t) acc.add(A, seg[t]);
    acc.write(A, o);
    return acc.bad;
}

// Ascending order of a segment, sorted in place when it is not (insertion
// sort: the segment is two ascending runs at worst).
__device__ __forceinline__ void sort_segment(uint32_t *seg, uint32_t len) {
    bool up = true;
    for (uint32_t t = 1; t < len; ++t) up &= seg[t - 1] < seg[t];
    if (up) return;
    for (uint32_t t = 1; t < len; ++t) {
        const uint32_t x = seg[t];
        uint32_t u = t;
        for (; u > 0 && seg[u - 1] > x; --u) seg[u] = seg[u - 1];
        seg[u] = x;
    }
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async8(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__global__ void __launch_bounds__(AG_THREADS, 5) k_agg_ops(const uint32_t *__restrict__ off, uint32_t *list,
                                                          AggIn A) {
    pdl_wait();
    extern __shared__ __align__(16) unsigned char ag_smem[];
    OpsWarp &W = reinterpret_cast<OpsWarp *>(ag_smem)[threadIdx.x / 32];
    const unsigned lane = lane_id();
    const bool ident = *A.nonident == 0;
    const float4 *rows = reinterpret_cast<const float4 *>(A.counters);
    // row index of kernel k, -1 for none (or for an index past the rows)
    auto row_of = [&](uint32_t k) -> int32_t {
        const int32_t j = ident ? (int32_t)k : A.ncu_idx[k];
        return j < A.M ? j : -1;
    };
    auto draw = [&]() -> unsigned {
        unsigned v = 0;
        if (lane == 0) v = atomicAdd(A.ctr, 1u);
        return v;
    };
    constexpr int PER = AG_CHUNK / 32;
    // the first chunk's offsets; afterwards the next chunk is drawn and its
    // offsets loaded while the current one runs
    int64_t o0 = (int64_t)__shfl_sync(0xffffffffu, draw(), 0) * AG_CHUNK;
    uint32_t oa[PER], ob[PER];
#pragma unroll
    for (int q = 0; q < PER; ++q) {
        const int64_t o = o0 + q * 32 + lane;
        oa[q] = o < A.n_ops ? off[o] : 0u;
        ob[q] = o < A.n_ops ? off[o + 1] : 0u;
    }
    while (o0 < A.n_ops) {
        const unsigned next_raw = draw();           // in flight during this chunk
        const int nchunk = A.n_ops - o0 < AG_CHUNK ? (int)(A.n_ops - o0) : AG_CHUNK;
        const uint32_t cbase = __shfl_sync(0xffffffffu, oa[0], 0);          // the chunk's list run
        const uint32_t cend = __shfl_sync(0xffffffffu, ob[(nchunk - 1) >> 5], (nchunk - 1) & 31);
        const uint32_t ctot = cend - cbase;
        const bool staged = ctot <= AG_STAGE;
        // lengths of the chunk's ops, counting sort by length (descending, capped)
        uint32_t bkt[PER];
        W.lcount[lane] = 0;
        __syncwarp();
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = q * 32 + (int)lane;
            const uint32_t len = i < nchunk ? ob[q] - oa[q] : 0u;
            bkt[q] = AG_LBUCKETS - 1 - (len < AG_LBUCKETS - 1 ? len : AG_LBUCKETS - 1);
            if (i < nchunk) atomicAdd(&W.lcount[bkt[q]], 1u);
        }
        if (staged)
            for (uint32_t i = lane; i < ctot; i += 32) W.L[i] = list[cbase + i];
        __syncwarp();
        {
            const unsigned x = W.lcount[lane];
            const unsigned inc = warp_inclusive_scan(x);
            W.lcount[lane] = inc - x;
        }
        __syncwarp();
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int i = q * 32 + (int)lane;
            if (i < nchunk) W.order[atomicAdd(&W.lcount[bkt[q]], 1u)] = (uint8_t)i;
            // each thread puts the segments of its own ops in ascending order
            const uint32_t len = i < nchunk ? ob[q] - oa[q] : 0u;
            if (len > AG_HUGE || (!staged && len > AG_SHORT_MAX)) {
                A.longs[atomicAdd(A.nlong, 1u)] = (uint32_t)(o0 + i);   // for the pieces pass
            } else if (len > 1) {
                if (staged) sort_segment(W.L + (oa[q] - cbase), len);
                else sort_segment(list + oa[q], len);
            }
        }
        __syncwarp();
        // the next chunk's offsets, in flight during the rounds
        const int64_t o1 = (int64_t)__shfl_sync(0xffffffffu, next_raw, 0) * AG_CHUNK;
        uint32_t na[PER], nb[PER];
#pragma unroll
        for (int q = 0; q < PER; ++q) {
            const int64_t o = o1 + q * 32 + lane;
            na[q] = o < A.n_ops ? off[o] : 0u;
            nb[q] = o < A.n_ops ? off[o + 1] : 0u;
        }
        for (int g = 0; g * 32 < nchunk; ++g) {
            const int i = g * 32 + (int)lane;
            // offsets of the op each lane walks, from the lane that holds them
            // (op il sits in register il >> 5 of lane il & 31)
            const int il = i < nchunk ? W.order[i] : 0;
            uint32_t sa = 0, sb = 0;
#pragma unroll
            for (int q = 0; q < PER; ++q) {
                const uint32_t xa = __shfl_sync(0xffffffffu, oa[q], il & 31);
                const uint32_t xb = __shfl_sync(0xffffffffu, ob[q], il & 31);
                if ((il >> 5) == q) { sa = xa; sb = xb; }
            }
            if (i >= nchunk) continue;
            const int64_t o = o0 + il;
            const uint32_t s0 = sa, len = sb - sa;
            if (len > AG_HUGE || (!staged && len > AG_SHORT_MAX)) continue;   // listed: k_agg_long_ops writes it
            const uint32_t *seg = staged ? W.L + (s0 - cbase) : list + s0;
            AccF acc;
            acc.init();
            if (len > 0) {
                // kernel t's row and duration land in slot t & 1 while kernel
                // t - 1 is added; row indices are loaded one step further ahead
                auto issue = [&](uint32_t t, uint32_t k, int32_t j) {
                    if (t < len) {
                        cp_async8(&W.dur[t & 1][lane], A.dur + k);
                        if (j >= 0) {
                            const float4 *src = rows + (int64_t)j * (NC / 4);
#pragma unroll
                            for (int c = 0; c < NC / 4; ++c) cp_async16(&W.row[t & 1][lane][c], src + c);
                        }
                    }
                    cp_async_commit();
                };
                const uint32_t k0 = seg[0], k1 = len > 1 ? seg[1] : 0u;
                const int32_t j0 = row_of(k0), j1 = len > 1 ? row_of(k1) : -1;
                uint32_t k2 = len > 2 ? seg[2] : 0u;
                int32_t j2 = len > 2 ? row_of(k2) : -1;
                issue(0, k0, j0);
                issue(1, k1, j1);
                int32_t js0 = j0, js1 = j1;           // row index of the kernel in each slot
                for (uint32_t t = 0; t < len; ++t) {
                    const uint32_t k3 = t + 3 < len ? seg[t + 3] : 0u;
                    const int32_t j3 = t + 3 < len ? row_of(k3) : -1;
                    cp_async_wait<1>();
                    const int32_t j = (t & 1) ? js1 : js0;
                    acc.accumulate(W.dur[t & 1][lane], j >= 0, W.row[t & 1][lane]);
                    issue(t + 2, k2, j2);
                    if (t & 1) js1 = j2; else js0 = j2;
                    k2 = k3;
                    j2 = j3;
                }
                cp_async_wait<0>();
            }
            // a null or infinite value poisons a sum: the op is listed for
            // k_agg_careful
            if (acc.clean()) acc.write(A, o, (int)len);
            else A.dirty[atomicAdd(A.ctr + 1, 1u)] = (uint32_t)o;
        }
        __syncwarp();
        o0 = o1;
#pragma unroll
        for (int q = 0; q < PER; ++q) { oa[q] = na[q]; ob[q] = nb[q]; }
    }
}

// The ops k_agg_ops listed as dirty: one thread each puts the segment in
// ascending kernel index (in place) and redoes it with Acc, which leaves
// nulls out and reports infinite values.  A separate pass keeps that rare,
// register-hungry path out of the ops pass.
__global__ void k_agg_careful(const uint32_t *__restrict__ off, uint32_t *list, AggIn A, DevStatus *st) {
    pdl_wait();
    int bad = 0;
    const unsigned n = A.ctr[1];
    for (unsigned e = blockIdx.x * blockDim.x + threadIdx.x; e < n; e += gridDim.x * blockDim.x) {
        const uint32_t o = A.dirty[e];
        const uint32_t s0 = off[o], len = off[o + 1] - s0;
        sort_segment(list + s0, len);
        bad |= op_careful(list + s0, len, A, o);
    }
    if (bad) set_err(st, ERR_INVALID);
}

// ------------------------------------------------------------------ host
// ------------------------------------------------------------------ long ops
// Ops the ops pass lists (longer than AG_HUGE, or longer than AG_SHORT_MAX
// in a chunk it could not stage; sorted by k_agg_sort_long or placed in order
// by a counting pass) are split into pieces of AG_PIECE kernels, so an
// operator with a very long segment (an Inductor fusion-map operator gathers
// every unattributed launch of its kernel name) is spread over many warps
// instead of holding one thread for its whole length.  Each lane adds a
// contiguous run of a piece in ascending kernel index with the careful
// accumulator; partials are combined by fixed trees of pairwise float-float
// additions (lane l takes lane l + 16, then l + 8, ...; a piece's partials in
// piece order), so results are reproducible, with an error bound of the
// longest run plus the pairwise steps.
__device__ __forceinline__ ff ff_pair_add(ff a, ff b) {
    const ff t = two_sum(a.hi, b.hi);
    return ff{t.hi, __fadd_rn(t.lo, __fadd_rn(a.lo, b.lo))};
}
__device__ __forceinline__ ff shfl_down_ff(ff v, int d) {
    return ff{__shfl_down_sync(0xffffffffu, v.hi, d), __shfl_down_sync(0xffffffffu, v.lo, d)};
}
__device__ __forceinline__ void acc_merge_down(Acc &a, int d) {
    const bool take = (int)lane_id() < d;
    const int kc = __shfl_down_sync(0xffffffffu, a.kc, d), mc = __shfl_down_sync(0xffffffffu, a.mc, d);
    const long long ds = __shfl_down_sync(0xffffffffu, a.dsum, d), da = __shfl_down_sync(0xffffffffu, a.dall, d);
    const unsigned seen = __shfl_down_sync(0xffffffffu, a.seen, d);
    const int bad = __shfl_down_sync(0xffffffffu, a.bad, d);
    if (take) {
        a.kc += kc; a.mc += mc; a.dsum += ds; a.dall += da; a.seen |= seen; a.bad |= bad;
    }
#pragma unroll
    for (int i = 0; i < N_SUM; ++i) {
        const ff x = shfl_down_ff(a.s[i], d);
        if (take) a.s[i] = ff_pair_add(a.s[i], x);
    }
#pragma unroll
    for (int i = 0; i < N_DW; ++i) {
        const ff x = shfl_down_ff(a.w[i], d);
        const long long nw = __shfl_down_sync(0xffffffffu, a.nanw[i], d);
        if (take) {
            a.w[i] = ff_pair_add(a.w[i], x);
            a.nanw[i] += nw;
        }
    }
#pragma unroll
    for (int i = 0; i < N_MAX; ++i) {
        const float x = __shfl_down_sync(0xffffffffu, a.mx[i], d);
        if (take) a.mx[i] = fmaxf(a.mx[i], x);
    }
}
// a += b, the same pairwise steps as acc_merge_down
__device__ __forceinline__ void acc_merge(Acc &a, const Acc &b) {
    a.kc += b.kc; a.mc += b.mc; a.dsum += b.dsum; a.dall += b.dall; a.seen |= b.seen; a.bad |= b.bad;
#pragma unroll
    for (int i = 0; i < N_SUM; ++i) a.s[i] = ff_pair_add(a.s[i], b.s[i]);
#pragma unroll
    for (int i = 0; i < N_DW; ++i) {
        a.w[i] = ff_pair_add(a.w[i], b.w[i]);
        a.nanw[i] += b.nanw[i];
    }
#pragma unroll
    for (int i = 0; i < N_MAX; ++i) a.mx[i] = fmaxf(a.mx[i], b.mx[i]);
}

// Piece offsets of the listed long ops, one block: poff[j] = pieces of the
// ops listed before j (an op longer than `huge` has ceil(len / AG_PIECE)
// pieces, a shorter one none); poff[nlong] = all pieces.
// info (may be NULL) receives {listed ops, pieces, longest huge op, kernels
// in huge ops, huge ops}; hop (with info) the huge ops in list order.
__global__ void __launch_bounds__(1024) k_agg_piece_offsets(const uint32_t *__restrict__ off,
                                                            const uint32_t *__restrict__ longs,
                                                            const unsigned *__restrict__ nlong, uint32_t huge,
                                                            uint32_t *__restrict__ poff, uint32_t *__restrict__ info,
                                                            uint32_t *__restrict__ hop) {
    pdl_wait();
    __shared__ uint32_t wbuf[33];
    const int64_t n = *nlong;
    uint32_t carry = 0, longest = 0, kern = 0, hcarry = 0;
    for (int64_t b = 0; b < n; b += 1024) {
        const int64_t j = b + threadIdx.x;
        uint32_t np = 0, o = 0;
        if (j < n) {
            o = longs[j];
            const uint32_t len = off[o + 1] - off[o];
            np = len > huge ? (len + AG_PIECE - 1) / AG_PIECE : 0u;
            if (np) {
                longest = len > longest ? len : longest;
                kern += len;
            }
        }
        uint32_t tot;
        const uint32_t ex = block_exclusive_scan<uint32_t>(np, wbuf, &tot);
        if (j < n) poff[j] = carry + ex;
        carry += tot;
        if (info) {
            uint32_t htot;
            const uint32_t hx = block_exclusive_scan<uint32_t>(np ? 1u : 0u, wbuf, &htot);
            if (np) hop[hcarry + hx] = o;
            hcarry += htot;
        }
    }
    if (threadIdx.x == 0) poff[n] = carry;
    if (info) {
        const uint32_t ksum = block_sum<uint32_t>(kern, wbuf);
        __shared__ uint32_t lmax;
        if (threadIdx.x == 0) lmax = 0;
        __syncthreads();
        atomicMax(&lmax, longest);
        __syncthreads();
        if (threadIdx.x == 0) {
            info[0] = (uint32_t)n;
            info[1] = carry;
            info[2] = lmax;
            info[3] = ksum;
            info[4] = hcarry;
        }
    }
}

// Huge ops' segments in ascending kernel index without sorting: with at most
// 256 huge ops, one counting pass over all kernels in index order, the digit
// being the index of the kernel's op among the huge ops, writes each such
// kernel to its op's segment at its rank among the op's kernels.
struct HugeDigit {
    const int32_t *rok;
    const uint32_t *r_op;
    int64_t R, n_ops;
    const uint32_t *hidx;        // [n_ops] index of a huge op among the huge ops, else 0xFFFFFFFF
    __device__ __forceinline__ unsigned operator()(int64_t k) const {
        const int32_t r = range_of(rok, r_op, k);
        if (r < 0 || r >= R) return RADIX_BINS;
        const uint32_t op = r_op[r];
        if ((int64_t)op >= n_ops) return RADIX_BINS;
        const uint32_t j = hidx[op];
        return j < RADIX_BINS ? j : (unsigned)RADIX_BINS;
    }
};
struct HugePlace {
    const uint32_t *hist;        // scanned digit-major histogram: hist[j * ntiles] = start of digit j
    int64_t ntiles;
    const uint32_t *hop, *off;   // the huge ops; the segment offsets
    uint32_t *list;
    __device__ __forceinline__ unsigned operator()(int64_t k, uint32_t dest, unsigned j) const {
        list[off[hop[j]] + (dest - hist[(int64_t)j * ntiles])] = (uint32_t)k;
        return 0u;
    }
    __device__ __forceinline__ void done(unsigned) const {}
};
__global__ void k_huge_index(const uint32_t *__restrict__ hop, int64_t n_huge, uint32_t *__restrict__ hidx) {
    pdl_wait();
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < n_huge; c += (int64_t)gridDim.x * blockDim.x)
        hidx[hop[c]] = (uint32_t)c;
}

// A lane's run of a piece with the fast accumulator: returns false when a
// null or infinite value took part (the caller redoes the run carefully),
// else the run's partial in careful form (every counter non-null).
__device__ __forceinline__ bool piece_fast(const AggIn &A, const uint32_t *seg, uint32_t l0, uint32_t l1, Acc &out) {
    AccF f;
    f.init();
#pragma unroll 4
    for (uint32_t t = l0; t < l1; ++t) {
        const uint32_t k = seg[t];
        const int32_t j = A.ncu_idx[k];
        const bool ok = j >= 0 && j < A.M;
        f.accumulate(A.dur[k], ok, reinterpret_cast<const float4 *>(A.counters + (int64_t)(ok ? j : 0) * NC));
    }
    if (!f.clean()) return false;
    out.kc = (int)(l1 - l0);
    out.mc = f.mc;
    out.dsum = f.dsum;
    out.dall = f.dall;
#pragma unroll
    for (int i = 0; i < N_SUM; ++i) out.s[i] = f.s[i];
#pragma unroll
    for (int i = 0; i < N_DW; ++i) {
        out.w[i] = f.w[i];
        out.nanw[i] = 0;
    }
#pragma unroll
    for (int i = 0; i < N_MAX; ++i) out.mx[i] = f.mx[i];
    out.seen = f.mc > 0 ? ALL_COUNTERS : 0u;
    out.bad = 0;
    out.terms = 0;
    return true;
}

// Pieces: one warp per AG_PIECE kernels of a huge op (lane l adds AG_PIECE /
// 32 consecutive kernels), the warp's 32 partials merged by the fixed tree,
// the piece's partial stored at its index.
__global__ void k_agg_pieces(const uint32_t *__restrict__ off, const uint32_t *__restrict__ list,
                             const uint32_t *__restrict__ longs, const unsigned *__restrict__ nlong,
                             const uint32_t *__restrict__ poff, AggIn A, Acc *__restrict__ part) {
    pdl_wait();
    const int64_t n = *nlong;
    const int64_t P = poff[n];
    const int64_t warp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const unsigned lane = lane_id();
    for (int64_t p = warp; p < P; p += nwarps) {
        int64_t lo = 0, hi = n;                   // the listed op: last j with poff[j] <= p
        while (hi - lo > 1) {
            const int64_t m = (lo + hi) >> 1;
            if ((int64_t)poff[m] <= p) lo = m; else hi = m;
        }
        const uint32_t o = longs[lo];
        const uint32_t s0 = off[o], len = off[o + 1] - s0;
        const uint32_t b0 = (uint32_t)(p - poff[lo]) * AG_PIECE;
        const uint32_t b1 = b0 + AG_PIECE < len ? b0 + AG_PIECE : len;
        const uint32_t per = AG_PIECE / 32;
        const uint32_t l0 = min(b0 + lane * per, b1), l1 = min(l0 + per, b1);
        Acc acc;
        if (!piece_fast(A, list + s0, l0, l1, acc)) {     // a null or infinite value: redo with null handling
            acc.init();
            for (uint32_t t = l0; t < l1; ++t) acc.add(A, list[s0 + t]);
        }
#pragma unroll 1
        for (int d = 16; d > 0; d >>= 1) acc_merge_down(acc, d);
        if (lane == 0) part[p] = acc;
    }
}

// Finish: one block per huge op merges its pieces' partials -- thread t takes
// pieces t, t + FIN_THREADS, ... in order, then each warp's fixed tree, then
// thread 0 takes the warps' partials in warp order -- and writes the record.
constexpr int FIN_THREADS = 256;
__global__ void __launch_bounds__(FIN_THREADS) k_agg_long_ops(const uint32_t *__restrict__ longs,
                                                              const unsigned *__restrict__ nlong,
                                                              const uint32_t *__restrict__ poff,
                                                              const Acc *__restrict__ part, int write_empty, AggIn A,
                                                              DevStatus *st) {
    pdl_wait();
    __shared__ Acc wpart[FIN_THREADS / 32];
    const int64_t n = *nlong;
    const unsigned lane = lane_id(), w = threadIdx.x >> 5;
    int bad = 0;
    for (int64_t q = blockIdx.x; q < n; q += gridDim.x) {
        if (poff[q + 1] == poff[q] && !write_empty) continue;   // not huge: the ops pass writes it
        const uint32_t o = longs[q];
        Acc acc;
        acc.init();
        for (uint32_t p = poff[q] + threadIdx.x; p < poff[q + 1]; p += FIN_THREADS) acc_merge(acc, part[p]);
#pragma unroll 1
        for (int d = 16; d > 0; d >>= 1) acc_merge_down(acc, d);
        if (lane == 0) wpart[w] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            Acc total = wpart[0];
            for (int v = 1; v < FIN_THREADS / 32; ++v) acc_merge(total, wpart[v]);
            total.write(A, o);
            bad |= total.bad;
        }
        __syncthreads();
    }
    if (bad) set_err(st, ERR_INVALID);
}

// Blocks of the ops pass: what stays resident, fewer for few ops.
static unsigned ops_grid(Ctx &c, int64_t O) {
    int sms = 0, per_sm = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_agg_ops, AG_THREADS, AG_SMEM);
    cudaGetLastError();
    const int64_t resident = (int64_t)std::max(1, sms) * std::max(1, per_sm);
    const int64_t need = (O + (int64_t)AG_WARPS * AG_CHUNK - 1) / ((int64_t)AG_WARPS * AG_CHUNK);
    return (unsigned)std::max<int64_t>(1, std::min(resident, need));
}

opattr_status do_aggregate(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                           const opattr_ncu *ncu, const int32_t *nidx, uint32_t n_ops,
                           const opattr_op_aggregates *out, opattr_totals *tot_out) {
    const int64_t K = kern->n, R = rng->n, M = ncu->n, O = n_ops;
    if (K < 0 || R < 0 || M < 0 || K >= (1ll << 31) || R >= (1ll << 31) || M >= (1ll << 31) || !out)
        return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->dur_ns || !nidx)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && !rok && R != K) return OPATTR_E_INVALID_ARG;     // one operator per kernel in rng->op_id
    if (R > 0 && !rng->op_id) return OPATTR_E_INVALID_ARG;
    if (M > 0 && !ncu->counters) return OPATTR_E_INVALID_ARG;
    if (O > 0 && (!out->kernel_count || !out->total_duration_ns || !out->matched_count || !out->agg))
        return OPATTR_E_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ncu->counters) & 15) != 0) return OPATTR_E_INVALID_ARG;

    Need nd;
    nd.add<uint32_t>(O + 1).add<uint32_t>(O + 1).add<uint32_t>(K).add<uint32_t>(K);
    nd.add<uint32_t>(O + 1).add<unsigned>(3).add<unsigned>(1).add<uint32_t>(O + 1);
    nd.add<uint32_t>(O + 1).add<Acc>(K / AG_PIECE + (K / (AG_SHORT_MAX + 1)) + 1);   // pieces per op, partials
    nd.add<uint32_t>(scan_scratch_elems(std::max<int64_t>(O + 1, radix_hist_elems(K))));
    nd.add<uint32_t>(O + 1).add<uint32_t>(radix_hist_elems(K)).add<uint32_t>(8);   // huge-op index, histogram, info
    nd.add<uint32_t>(O + 1);                                                         // huge ops
    opattr_status st = ensure_arena(c, nd.bytes + 4096);
    if (st) return st;
    Arena a(c);
    // with the enclosure's verdict pending (a join) the status block keeps it:
    // the enclosure's reset left the aggregation's slots at zero
    if (!c.enclose_pending && (st = reset_status(c))) return st;
    uint32_t *cnt = a.take<uint32_t>(O + 1), *off = a.take<uint32_t>(O + 1);
    // tmp holds each kernel's slot among its op's kernels until the list is
    // placed, then serves the segment sorts
    uint32_t *list = a.take<uint32_t>(K), *tmp = a.take<uint32_t>(K), *longs = a.take<uint32_t>(O + 1);
    // ctr[0] next chunk, ctr[1] ops listed dirty, ctr[2] (nlong) ops listed long:
    // the two counts come back together
    unsigned *ctr = a.take<unsigned>(3);
    unsigned *nlong = ctr ? ctr + 2 : nullptr;
    unsigned *nonident = a.take<unsigned>(1);
    uint32_t *dirty = a.take<uint32_t>(O + 1);
    uint32_t *npc = a.take<uint32_t>(O + 1);
    Acc *partials = a.take<Acc>(K / AG_PIECE + (K / (AG_SHORT_MAX + 1)) + 1);
    if (!npc || !partials) return OPATTR_E_OOM;
    cudaMemsetAsync(ctr, 0, 3 * sizeof(unsigned), c.stream);
    uint32_t *part = a.take<uint32_t>(scan_scratch_elems(std::max<int64_t>(O + 1, radix_hist_elems(K))));
    uint32_t *hidx = a.take<uint32_t>(O + 1), *hhist = a.take<uint32_t>(radix_hist_elems(K));
    uint32_t *info = a.take<uint32_t>(8), *hop = a.take<uint32_t>(O + 1);
    if (!hidx || !hhist || !info || !hop) return OPATTR_E_OOM;
    if (!cnt || !off || !list || !tmp || !longs || !nlong || !part || !nonident || !dirty) return OPATTR_E_OOM;
    cudaMemsetAsync(cnt, 0, sizeof(uint32_t) * (O + 1), c.stream);
    cudaMemsetAsync(nonident, 0, sizeof(unsigned), c.stream);
    int sms = 0;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
    // runs long enough to keep most segments in one warp, short enough that
    // the grid is one wave of resident warps (five blocks of eight per SM)
    const int64_t warps = (int64_t)std::max(1, sms) * 40;
    const int64_t run = std::min<int64_t>(AF_RUN, std::max<int64_t>(32, ((K + warps - 1) / warps + 31) / 32 * 32));
    if (K > 0)
        launch(c, "agg_count", rok ? k_agg_count<false> : k_agg_count<true>,
               dim3(grid_for(K, 256 / 32 * run, 65535)), dim3(256), 0, kern->dur_ns, rok, nidx, rng->op_id, K, R, M,
               O, cnt, tmp, run, (int)(c.in_join && c.rows_identity), nonident, c.d_status);
    AggIn in;
    in.dur = kern->dur_ns;
    in.ncu_idx = nidx;
    in.counters = ncu->counters;
    in.M = M;
    in.n_ops = O;
    in.ctr = ctr;
    in.dirty = dirty;
    in.longs = longs;
    in.nlong = nlong;
    in.nonident = nonident;
    in.out = *out;
    bool status_fresh = false;        // no launch since the last status read
    if (O > 0) {
        scan_exclusive_u32(c, cnt, off, O + 1, part, nullptr);
        if (K > 0)
            launch(c, "agg_place", rok ? k_agg_place<false> : k_agg_place<true>,
                   dim3(grid_for(K, 256 * 4, REDUCE_GRID)), dim3(256), 0, rok, rng->op_id, K, R, O,
                   (const uint32_t *)off, (const uint32_t *)tmp, list);
        static unsigned attr_done = 0;
        if (c.device < 32 && !(attr_done & (1u << c.device))) {
            cudaFuncSetAttribute(k_agg_ops, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)AG_SMEM);
            attr_done |= 1u << c.device;
        }
        launch(c, "agg_ops", k_agg_ops, dim3(ops_grid(c, O)), dim3(AG_THREADS), AG_SMEM,
               (const uint32_t *)off, list, in);
        // the ops the pass left: listed with a null or infinite value (redone
        // by k_agg_careful), long ones (the pieces pass); both
        // counts come back with the status
        const SmallCopy counts{c.h_levels, ctr + 1, 2 * sizeof(uint32_t)};
        if ((st = read_status(c, 1, &counts))) return st;
        const uint32_t n_dirty = c.h_levels[0], n_long = c.h_levels[1];
        status_fresh = n_dirty == 0 && n_long == 0;
        if (n_dirty > 0)
            launch(c, "agg_careful", k_agg_careful, dim3(std::max(1, sms)), dim3(128), 0, (const uint32_t *)off, list,
                   in, c.d_status);
        uint32_t pieces = 0, longest = 0, n_huge = 0;
        if (n_long > 0) {
            launch(c, "agg_piece_offsets", k_agg_piece_offsets, dim3(1), dim3(1024), 0, (const uint32_t *)off,
                   (const uint32_t *)longs, (const unsigned *)nlong, 0u, npc, info, hop);
            const SmallCopy pinfo{c.h_levels, info, 5 * sizeof(uint32_t)};
            if ((st = read_status(c, 1, &pinfo))) return st;
            pieces = c.h_levels[1];
            longest = c.h_levels[2];
            n_huge = c.h_levels[4];
        }
        if (pieces > 0) {
            if (n_huge <= (uint32_t)RADIX_BINS && longest > AG_BLOCK_SORT_MAX && K > 0) {
                // very long segments: placed in kernel order by one counting pass
                cudaMemsetAsync(hidx, 0xFF, sizeof(uint32_t) * (O + 1), c.stream);
                launch(c, "huge_index", k_huge_index, dim3(grid_for(n_huge, 256, 4096)), dim3(256), 0,
                       (const uint32_t *)hop, (int64_t)n_huge, hidx);
                const HugeDigit dg{rok, rng->op_id, R, O, hidx};
                const uint32_t *hoffs = digit_offsets(c, dg, K, hhist, part);
                const int64_t ntiles = (K + RADIX_TILE - 1) / RADIX_TILE;
                digit_rank(c, "huge_place", dg, K, hoffs,
                           HugePlace{hoffs, ntiles, (const uint32_t *)hop, (const uint32_t *)off, list});
            } else {
                launch(c, "agg_sort_long", k_agg_sort_long, dim3(2 * std::max(1, sms)), dim3(SL_THREADS), 0,
                       (const uint32_t *)off, (const uint32_t *)longs, (const unsigned *)nlong, 2u,
                       0xFFFFFFFFu, list, tmp);
            }
            launch(c, "agg_pieces", k_agg_pieces, dim3(4 * std::max(1, sms)), dim3(256), 0, (const uint32_t *)off,
                   (const uint32_t *)list, (const uint32_t *)longs, (const unsigned *)nlong, (const uint32_t *)npc,
                   in, partials);
            launch(c, "agg_long_ops", k_agg_long_ops, dim3(2 * std::max(1, sms)), dim3(FIN_THREADS), 0,
                   (const uint32_t *)longs, (const unsigned *)nlong, (const uint32_t *)npc,
                   (const Acc *)partials, 0, in, c.d_status);
        }
    }
    if (!status_fresh && (st = read_status(c))) return st;
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
    if (tot_out) *tot_out = T;
    return OPATTR_OK;
}

}  // namespace opattr

namespace opattr {

// ------------------------------------------------------------------ class roll-up
// The per-operator records of Eq. (1) rolled up to operator classes (the
// per-class breakdown of the case studies): every attributed kernel whose
// operator has a class is aggregated with the other kernels of that class.
// Few, large groups: a stable radix sort of the kernels by class key (kernel
// index order kept within a class) replaces the placement and the segment sort,
// and every class is accumulated by pieces.
__global__ void k_class_check(const uint32_t *__restrict__ class_of_op, int64_t n_ops, uint32_t n_classes,
                              DevStatus *st) {
    pdl_wait();
    int bad = 0;
    for (int64_t o = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; o < n_ops; o += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t c = class_of_op[o];
        bad |= c >= n_classes && c != OPATTR_OP_NONE;
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
}
// key = class of the kernel's operator, n_classes when it has none; counts
// per class (in a block histogram in shared memory when there are at most
// CK_SMEM classes, flushed once per block; else one global atomic per class
// and warp).
constexpr int CK_SMEM = 4096;
__global__ void k_class_keys(const int32_t *__restrict__ rok, const uint32_t *__restrict__ r_op, int64_t K, int64_t R,
                             int64_t n_ops, const uint32_t *__restrict__ class_of_op, uint32_t n_classes,
                             uint32_t *__restrict__ key, uint32_t *__restrict__ cnt) {
    pdl_wait();
    __shared__ uint32_t h[CK_SMEM];
    const bool local = n_classes <= (uint32_t)CK_SMEM;
    if (local)
        for (uint32_t i = threadIdx.x; i < n_classes; i += blockDim.x) h[i] = 0;
    __syncthreads();
    uint32_t *dst = local ? h : cnt;
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k - threadIdx.x < K;
         k += (int64_t)gridDim.x * blockDim.x) {
        uint32_t c = n_classes;
        if (k < K) {
            const int32_t r = range_of(rok, r_op, k);
            if (r >= 0 && r < R) {
                const uint32_t op = r_op[r];
                if ((int64_t)op < n_ops) {
                    const uint32_t x = class_of_op[op];
                    if (x < n_classes) c = x;
                }
            }
            key[k] = c;
        }
        const unsigned peers = __match_any_sync(0xffffffffu, c);
        if (k < K && c < n_classes && (peers & lanemask_lt()) == 0) atomicAdd(&dst[c], (unsigned)__popc(peers));
    }
    if (local) {
        __syncthreads();
        for (uint32_t i = threadIdx.x; i < n_classes; i += blockDim.x)
            if (h[i]) atomicAdd(&cnt[i], h[i]);
    }
}
__global__ void k_iota_u32(uint32_t *dst, int64_t n, unsigned *count) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = (uint32_t)i;
    if (blockIdx.x == 0 && threadIdx.x == 0) *count = (unsigned)n;
}

opattr_status do_rollup(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                        const opattr_ncu *ncu, const int32_t *nidx, uint32_t n_ops, const uint32_t *class_of_op,
                        uint32_t n_classes, const opattr_op_aggregates *out) {
    const int64_t K = kern->n, R = rng->n, M = ncu->n, O = n_ops, C = n_classes;
    if (K < 0 || R < 0 || M < 0 || K >= (1ll << 31) || R >= (1ll << 31) || M >= (1ll << 31) || !out)
        return OPATTR_E_INVALID_ARG;
    if (C > (1 << 24)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->dur_ns || !nidx)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && !rok && R != K) return OPATTR_E_INVALID_ARG;
    if (R > 0 && !rng->op_id) return OPATTR_E_INVALID_ARG;
    if (O > 0 && !class_of_op) return OPATTR_E_INVALID_ARG;
    if (M > 0 && !ncu->counters) return OPATTR_E_INVALID_ARG;
    if (C > 0 && (!out->kernel_count || !out->total_duration_ns || !out->matched_count || !out->agg))
        return OPATTR_E_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(ncu->counters) & 15) != 0) return OPATTR_E_INVALID_ARG;

    const int64_t maxp = K / AG_PIECE + C + 1;
    Need nd;
    for (int i = 0; i < 4; ++i) nd.add<uint32_t>(K);
    nd.add<uint32_t>(radix_hist_elems(K)).add<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), C + 2)));
    nd.add<uint32_t>(C + 2).add<uint32_t>(C + 2).add<uint32_t>(C + 1).add<uint32_t>(C + 1).add<unsigned>(1);
    nd.add<Acc>(maxp);
    opattr_status st = ensure_arena(c, nd.bytes + 4096);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;
    uint32_t *k0 = a.take<uint32_t>(K), *v0 = a.take<uint32_t>(K), *k1 = a.take<uint32_t>(K), *v1 = a.take<uint32_t>(K);
    uint32_t *hist = a.take<uint32_t>(radix_hist_elems(K));
    uint32_t *part = a.take<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), C + 2)));
    uint32_t *cnt = a.take<uint32_t>(C + 2), *off = a.take<uint32_t>(C + 2);
    uint32_t *cls = a.take<uint32_t>(C + 1), *poff = a.take<uint32_t>(C + 1);
    unsigned *ncls = a.take<unsigned>(1);
    Acc *partials = a.take<Acc>(maxp);
    if (!k0 || !v0 || !k1 || !v1 || !hist || !part || !cnt || !off || !cls || !poff || !ncls || !partials)
        return OPATTR_E_OOM;
    if (O > 0)
        launch(c, "class_check", k_class_check, dim3(grid_for(O, 256, REDUCE_GRID)), dim3(256), 0, class_of_op, O,
               n_classes, c.d_status);
    cudaMemsetAsync(cnt, 0, sizeof(uint32_t) * (C + 2), c.stream);
    uint32_t *list = nullptr;
    if (K > 0) {
        launch(c, "class_keys", k_class_keys, dim3(grid_for(K, 256, REDUCE_GRID)), dim3(256), 0, rok, rng->op_id, K, R,
               O, class_of_op, n_classes, k0, cnt);
        uint32_t *ko;
        radix_sort_pairs<uint32_t>(c, k0, v0, k1, v1, K, bits_for((uint64_t)C), true, hist, part, &ko, &list);
    }
    scan_exclusive_u32(c, cnt, off, C + 1, part, nullptr);           // off[C] = kernels with a class
    if (C > 0) {
        AggIn in;
        in.dur = kern->dur_ns;
        in.ncu_idx = nidx;
        in.counters = ncu->counters;
        in.M = M;
        in.n_ops = C;
        in.ctr = nullptr;
        in.dirty = nullptr;
        in.longs = nullptr;
        in.nlong = nullptr;
        in.nonident = nullptr;
        in.out = *out;
        int sms = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, c.device);
        launch(c, "class_iota", k_iota_u32, dim3(grid_for(C, 256, 4096)), dim3(256), 0, cls, C, ncls);
        launch(c, "agg_piece_offsets", k_agg_piece_offsets, dim3(1), dim3(1024), 0, (const uint32_t *)off,
               (const uint32_t *)cls, (const unsigned *)ncls, 0u, poff, (uint32_t *)nullptr, (uint32_t *)nullptr);
        if (K > 0)
            launch(c, "agg_pieces", k_agg_pieces, dim3(4 * std::max(1, sms)), dim3(256), 0, (const uint32_t *)off,
                   (const uint32_t *)list, (const uint32_t *)cls, (const unsigned *)ncls, (const uint32_t *)poff, in,
                   partials);
        launch(c, "class_records", k_agg_long_ops, dim3(2 * std::max(1, sms)), dim3(FIN_THREADS), 0,
               (const uint32_t *)cls,
               (const unsigned *)ncls, (const uint32_t *)poff, (const Acc *)partials, 1, in, c.d_status);
    }
    if ((st = read_status(c))) return st;
    if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    return OPATTR_OK;
}

}  // namespace opattr
