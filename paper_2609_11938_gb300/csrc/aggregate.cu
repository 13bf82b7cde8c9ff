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
struct Acc {
    long long kc, dsum, mc;
    ff s[N_SUM];
    ff w[N_DW];
    long long den[N_DW];
    float mx[N_MAX];
    unsigned seen;      // bit c: counter c had a non-null value
    int bad;            // an infinite counter was seen

    __device__ __forceinline__ void init() {
        kc = dsum = mc = 0;
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) s[i] = ff{0.f, 0.f};
#pragma unroll
        for (int i = 0; i < N_DW; ++i) { w[i] = ff{0.f, 0.f}; den[i] = 0; }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) mx[i] = -INFINITY;
        seen = 0;
        bad = 0;
    }

    __device__ __forceinline__ void add(const AggIn &A, int64_t k) {
        const long long d = A.dur[k];
        kc++;
        dsum += d;
        const int32_t j = A.ncu_idx[k];
        if (j < 0) return;
        mc++;
        const float4 *row = reinterpret_cast<const float4 *>(A.counters + (int64_t)j * NC);
        float v[NC];
#pragma unroll
        for (int q = 0; q < NC / 4; ++q) {
            float4 x = __ldg(row + q);
            v[4 * q] = x.x; v[4 * q + 1] = x.y; v[4 * q + 2] = x.z; v[4 * q + 3] = x.w;
        }
        const ff dd = ff_from_i64(d);
#pragma unroll
        for (int i = 0; i < N_SUM; ++i) {
            const int c = i == 0 ? 0 : i == 1 ? 1 : i == 2 ? 2 : i == 3 ? 10 : i == 4 ? 14 : 18;
            const unsigned u = __float_as_uint(v[c]);
            if ((u & 0x7F800000u) == 0x7F800000u) { bad |= (u & 0x7FFFFFu) == 0; continue; }
            seen |= 1u << c;
            ff_add(s[i], v[c], 0.f);
        }
#pragma unroll
        for (int i = 0; i < N_DW; ++i) {
            const int c = i < 7 ? 3 + i : (i < 10 ? 4 + i : 5 + i);   // 3..9, 11..13, 15..16
            const unsigned u = __float_as_uint(v[c]);
            if ((u & 0x7F800000u) == 0x7F800000u) { bad |= (u & 0x7FFFFFu) == 0; continue; }
            seen |= 1u << c;
            ff p = ff_mul_f(v[c], dd);
            ff_add(w[i], p.hi, p.lo);
            den[i] += d;
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) {
            const int c = i == 0 ? 17 : 19;
            const unsigned u = __float_as_uint(v[c]);
            if ((u & 0x7F800000u) == 0x7F800000u) { bad |= (u & 0x7FFFFFu) == 0; continue; }
            seen |= 1u << c;
            mx[i] = fmaxf(mx[i], v[c]);
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
        for (int i = 0; i < N_SUM; ++i) {
            const int c = i == 0 ? 0 : i == 1 ? 1 : i == 2 ? 2 : i == 3 ? 10 : i == 4 ? 14 : 18;
            agg[(int64_t)c * n + op] = ((seen >> c) & 1u) ? ff_to_f64(s[i]) : qnan;
        }
#pragma unroll
        for (int i = 0; i < N_DW; ++i) {
            const int c = i < 7 ? 3 + i : (i < 10 ? 4 + i : 5 + i);
            agg[(int64_t)c * n + op] = (((seen >> c) & 1u) && den[i] > 0) ? ff_div_i64_to_f64(w[i], den[i]) : qnan;
        }
#pragma unroll
        for (int i = 0; i < N_MAX; ++i) {
            const int c = i == 0 ? 17 : 19;
            agg[(int64_t)c * n + op] = ((seen >> c) & 1u) ? f32_to_f64_bits(mx[i]) : qnan;
        }
    }
};

// ------------------------------------------------------------------ checks and totals
// Per kernel: duration >= 0, range index in [-1, R), an attributed range is an
// operator below n_ops, row index in [-1, M).  Totals: all / attributed time,
// attributed and matched kernel counts.
__global__ void k_agg_check_kernels(const int64_t *__restrict__ dur, const int32_t *__restrict__ rok,
                                    const int32_t *__restrict__ nidx, const uint32_t *__restrict__ r_op, int64_t K,
                                    int64_t R, int64_t M, int64_t n_ops, DevStatus *st) {
    unsigned long long tot = 0, att = 0, natt = 0, nmatch = 0;
    int bad = 0;
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x) {
        long long d = dur[k];
        int32_t r = rok[k], j = nidx[k];
        if (d < 0 || r < -1 || r >= R || j < -1 || j >= M) { bad = 1; continue; }
        tot += (unsigned long long)d;
        if (r >= 0) {
            uint32_t op = r_op[r];
            if ((int64_t)op >= n_ops) { bad = 1; continue; }
            att += (unsigned long long)d;
            natt++;
            nmatch += j >= 0;
        }
    }
    tot = warp_sum(tot);
    att = warp_sum(att);
    natt = warp_sum(natt);
    nmatch = warp_sum(nmatch);
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
    if (lane_id() == 0) {
        if (tot) atomicAdd(&st->cnt[C_TOTAL_NS], tot);
        if (att) atomicAdd(&st->cnt[C_ATTR_NS], att);
        if (natt) atomicAdd(&st->cnt[C_ATTR_K], natt);
        if (nmatch) atomicAdd(&st->cnt[C_MATCHED_K], nmatch);
    }
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
constexpr int AGG_THREADS = 256;
constexpr int AGG_TILE = 1024;               // kernels per tile
constexpr int AGG_SLOTS = 512;               // owned ranges handled per pass
constexpr int AGG_WARPS = AGG_THREADS / 32;
constexpr int AGG_PER_WARP = AGG_TILE / AGG_WARPS;

// band[t] = number of ranges with start <= T(t * AGG_TILE - 1), band[0] = 0,
// band[nt] = R: tile t owns ranges [band[t], band[t+1]).
__global__ void k_band_table(const int64_t *__restrict__ k_start, int64_t K, const int64_t *__restrict__ r_start,
                             int64_t R, int64_t nt, int64_t *__restrict__ band) {
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t <= nt; t += (int64_t)gridDim.x * blockDim.x) {
        if (t == 0) { band[0] = 0; continue; }
        if (t == nt) { band[nt] = R; continue; }
        long long b = k_start[t * AGG_TILE - 1];
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
    const int64_t *k_start;
    const int32_t *rok;
    int64_t K;
    const int64_t *r_end;
    const uint32_t *r_op;
    const int64_t *band;
    DevStatus *st;
};

struct OwnSmem {
    int32_t rok[AGG_TILE];
    uint16_t klist[AGG_TILE];
    uint16_t wcnt[AGG_WARPS][AGG_SLOTS];
    uint16_t soff[AGG_SLOTS + 1];
    uint32_t wbuf[33];
    unsigned long long seen;
    int bad;
};

__global__ void __launch_bounds__(AGG_THREADS) k_agg_owned(OwnArgs A) {
    __shared__ OwnSmem S;
    const int64_t t = blockIdx.x;
    const int64_t k0 = t * AGG_TILE;
    const int64_t kn = A.K - k0 < AGG_TILE ? A.K - k0 : AGG_TILE;
    const int64_t k1 = k0 + kn;
    const int64_t ra = A.band[t], rb = A.band[t + 1];
    const long long t_next = k1 < A.K ? A.k_start[k1] : LLONG_MAX;
    const unsigned w = threadIdx.x >> 5, lane = lane_id(), lt = lanemask_lt();
    for (int i = threadIdx.x; i < AGG_TILE; i += AGG_THREADS) S.rok[i] = i < kn ? A.rok[k0 + i] : -1;
    if (threadIdx.x == 0) { S.seen = 0; S.bad = 0; }
    unsigned long long seen = 0;
    int bad = 0;

    for (int64_t ca = ra; ca < rb; ca += AGG_SLOTS) {
        const int64_t cb = rb - ca < AGG_SLOTS ? rb : ca + AGG_SLOTS;
        const int nslot = (int)(cb - ca);
        for (int i = threadIdx.x; i < AGG_WARPS * AGG_SLOTS; i += AGG_THREADS) (&S.wcnt[0][0])[i] = 0;
        __syncthreads();
        // stable in-tile ranking by slot: warp w owns kernels [w*128, w*128+128)
        uint16_t rank[AGG_PER_WARP / 32];
        int slot_of[AGG_PER_WARP / 32];
#pragma unroll
        for (int it = 0; it < AGG_PER_WARP / 32; ++it) {
            int i = w * AGG_PER_WARP + it * 32 + lane;
            int32_t r = S.rok[i];
            int sl = (r >= ca && r < cb) ? (int)(r - ca) : AGG_SLOTS;
            unsigned peers = __match_any_sync(0xffffffffu, sl);
            unsigned before = sl < AGG_SLOTS ? S.wcnt[w][sl] : 0u;
            __syncwarp();
            if (sl < AGG_SLOTS && (peers & lt) == 0) S.wcnt[w][sl] = (uint16_t)(before + __popc(peers));
            __syncwarp();
            rank[it] = (uint16_t)(before + __popc(peers & lt));
            slot_of[it] = sl;
        }
        __syncthreads();
        // per slot: exclusive prefix over warps, then over slots
        for (int b = 0; b < AGG_SLOTS; b += AGG_THREADS) {
            int sl = b + threadIdx.x;
            unsigned tot = 0;
#pragma unroll
            for (int q = 0; q < AGG_WARPS; ++q) {
                unsigned x = S.wcnt[q][sl];
                S.wcnt[q][sl] = (uint16_t)tot;
                tot += x;
            }
            unsigned all;
            unsigned ex = block_exclusive_scan<unsigned>(tot, S.wbuf, &all);
            unsigned carry = b == 0 ? 0u : S.soff[b];
            __syncthreads();
            S.soff[sl] = (uint16_t)(carry + ex);
            if (threadIdx.x == AGG_THREADS - 1) S.soff[b + AGG_THREADS] = (uint16_t)(carry + ex + tot);
            __syncthreads();
        }
#pragma unroll
        for (int it = 0; it < AGG_PER_WARP / 32; ++it) {
            int sl = slot_of[it];
            if (sl < AGG_SLOTS) {
                int i = w * AGG_PER_WARP + it * 32 + lane;
                S.klist[S.soff[sl] + S.wcnt[w][sl] + rank[it]] = (uint16_t)i;
            }
        }
        __syncthreads();
        // one thread per owned range: its kernels in this tile, then beyond it
        for (int sl = threadIdx.x; sl < nslot; sl += AGG_THREADS) {
            const int64_t r = ca + sl;
            const uint32_t op = A.r_op[r];
            if ((int64_t)op >= A.in.n_ops) continue;             // not an operator range
            Acc acc;
            acc.init();
            for (int q = S.soff[sl]; q < S.soff[sl + 1]; ++q) acc.add(A.in, k0 + S.klist[q]);
            const long long e = A.r_end[r];
            if (e >= t_next) {
                for (int64_t k = k1; k < A.K; ++k) {
                    if (A.k_start[k] > e) break;
                    if (A.rok[k] == (int32_t)r) acc.add(A.in, k);
                }
            }
            acc.write(A.in, op);
            seen += (unsigned long long)acc.kc;
            bad |= acc.bad;
        }
        __syncthreads();
    }
    seen = warp_sum(seen);
    if (lane == 0 && seen) atomicAdd(&S.seen, seen);
    if (__any_sync(0xffffffffu, bad) && lane == 0) S.bad = 1;
    __syncthreads();
    if (threadIdx.x == 0) {
        if (S.seen) atomicAdd(&A.st->cnt[C_AGG_SEEN], S.seen);
        if (S.bad) set_err(A.st, ERR_INVALID);
    }
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

    const int64_t nt = (K + AGG_TILE - 1) / AGG_TILE;
    Need nd;
    nd.add<unsigned>((O + 31) / 32 + 1).add<int64_t>(nt + 1);
    for (int i = 0; i < 7; ++i) nd.add<uint32_t>(K);
    nd.add<uint32_t>(radix_hist_elems(K)).add<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), K)));
    opattr_status st = ensure_arena(c, nd.bytes + 4096);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;
    unsigned *bitmap = a.take<unsigned>((O + 31) / 32 + 1);
    int64_t *band = a.take<int64_t>(nt + 1);
    if (!bitmap || !band) return OPATTR_E_OOM;
    cudaMemsetAsync(bitmap, 0, sizeof(unsigned) * ((O + 31) / 32 + 1), c.stream);
    if (K > 0) {
        launch(c, "agg_check_kernels", k_agg_check_kernels, dim3(grid_for(K, 256, 65535)), dim3(256), 0, kern->dur_ns,
               rok, nidx, rng->op_id, K, R, M, O, c.d_status);
        check_kernel_order(c, kern->stream, kern->start_ns, K);
    }
    if (R > 0)
        launch(c, "agg_check_ranges", k_agg_check_ranges, dim3(grid_for(R, 256, 65535)), dim3(256), 0, rng->start_ns,
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
        A.k_start = kern->start_ns;
        A.rok = rok;
        A.K = K;
        A.r_end = rng->end_ns;
        A.r_op = rng->op_id;
        A.band = band;
        A.st = c.d_status;
        launch(c, "agg_owned", k_agg_owned, dim3((unsigned)nt), dim3(AGG_THREADS), 0, A);
        launch(c, "agg_fill_unreferenced", k_agg_fill_unreferenced, dim3(grid_for(O, 256, 65535)), dim3(256), 0,
               (const unsigned *)bitmap, in);
        if ((st = read_status(c))) return st;
        if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
        fast = c.h_status->cnt[C_AGG_SEEN] == c.h_status->cnt[C_ATTR_K];
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
