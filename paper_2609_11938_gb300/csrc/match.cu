// match.cu -- Algorithm 1 (invocation-order matching, Sec. 3.3) and layer
// deduplication broadcast (Sec. 3.7) on the GPU.
//
// Fast path.  When the replayed kernels, in time order, carry exactly the
// names of the ncu rows in array order, launch i pairs with row i and no
// ordinal is computed: one pass compares the two name arrays and writes the
// identity.  Exports in time order with ncu replaying the same launches hit
// this path.  With per-stream rows (the rows of each stream in launch order,
// streams one after another) the same test runs on the replayed kernels and
// the rows each partitioned stably by stream.
//
// General path.  Ordinals come from stable radix sorts: replayed kernels in
// time order sorted by name give o(k) = position - start of the name's run;
// ncu rows in array order sorted by name give the rows of each name in
// launch order.  The join is row = rows_of_name[o(k)], subject to the
// mismatch mode.  Dedup positions come the same way from a stable sort of
// layer-tagged kernels by layer id.
#include <algorithm>

#include "sort.cuh"
#include "util.cuh"

namespace opattr {

// ------------------------------------------------------------------ fast path
// Whether the identity pass may use 16-byte accesses (every array aligned).
static int identity_vec(const void *kname, const void *nname, const void *out_idx, const void *out_kind) {
    auto al = [](const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
    return al(kname, 16) && al(nname, 16) && al(out_idx, 16) && al(out_kind, 4);
}
__global__ void k_match_identity(const uint32_t *__restrict__ kname, const uint32_t *__restrict__ nname, int64_t n,
                                 int32_t *__restrict__ out_idx, uint8_t *__restrict__ out_kind, int vec,
                                 DevStatus *st) {
    pdl_wait();
    constexpr int U = 4;                    // elements per thread per round, loads issued together
    int bad = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x * U;
    for (int64_t base = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * U; base < n; base += stride) {
        if (vec && base + U <= n) {         // 16-byte loads and stores
            const uint4 a = *reinterpret_cast<const uint4 *>(kname + base);
            const uint4 b = *reinterpret_cast<const uint4 *>(nname + base);
            bad |= (a.x != b.x) | (a.y != b.y) | (a.z != b.z) | (a.w != b.w);
            const int32_t i0 = (int32_t)base;
            *reinterpret_cast<int4 *>(out_idx + base) = make_int4(i0, i0 + 1, i0 + 2, i0 + 3);
            if (out_kind) *reinterpret_cast<uint32_t *>(out_kind + base) = 0x01010101u;
            continue;
        }
        uint32_t a[U], b[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            a[u] = base + u < n ? kname[base + u] : 0u;
            b[u] = base + u < n ? nname[base + u] : 0u;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (base + u >= n) continue;
            bad |= a[u] != b[u];
            out_idx[base + u] = (int32_t)(base + u);
            if (out_kind) out_kind[base + u] = 1;
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_flag(st, F_NAMES_DIFFER);
}

void launch_identity_match(Ctx &c, const uint32_t *kname, const uint32_t *nname, int64_t K, int32_t *out_idx,
                           uint8_t *out_kind) {
    launch(c, "match_identity", k_match_identity, dim3(grid_for(K, 256 * 16, REDUCE_GRID)), dim3(256), 0, kname,
           nname, K, out_idx, out_kind, identity_vec(kname, nname, out_idx, out_kind), c.d_status);
}

// replayed kernels in time order (list rk) against rows 0..n-1
__global__ void k_match_identity_list(const uint32_t *__restrict__ rk, const uint32_t *__restrict__ kname,
                                      const uint32_t *__restrict__ nname, int64_t n, int32_t *__restrict__ out_idx,
                                      uint8_t *__restrict__ out_kind, DevStatus *st) {
    pdl_wait();
    int bad = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t k = rk[i];
        bad |= kname[k] != nname[i];
        out_idx[k] = (int32_t)i;
        if (out_kind) out_kind[k] = 1;
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_flag(st, F_NAMES_DIFFER);
}

// Per-stream rows.  Replayed kernel j (kernel rk[j], or j when rk is null)
// takes position dest of the replayed kernels partitioned stably by stream;
// the row at that position of the rows partitioned the same way is pn[dest].
// The pairing holds when name and stream agree everywhere; name ids must
// also fit in 24 bits, as (name, stream) keys require.
struct StreamDigit {
    const uint32_t *rk;
    const uint8_t *stream;
    __device__ __forceinline__ unsigned operator()(int64_t j) const { return stream[rk ? rk[j] : (uint32_t)j]; }
};
struct StreamPairs {
    const uint32_t *rk, *pn, *kname, *nname;
    const uint8_t *kstream, *nstream;
    int32_t *out_idx;
    uint8_t *out_kind;
    DevStatus *st;
    __device__ __forceinline__ unsigned operator()(int64_t j, uint32_t dest, unsigned) const {
        const uint32_t k = rk ? rk[j] : (uint32_t)j;
        const uint32_t r = pn[dest];
        const uint32_t x = kname[k], y = nname[r];
        out_idx[k] = (int32_t)r;
        if (out_kind) out_kind[k] = 1;
        return (x != y || kstream[k] != nstream[r] ? 1u : 0u) | ((x | y) >> 24 != 0 ? 2u : 0u);
    }
    __device__ __forceinline__ void done(unsigned bits) const {
        if (__any_sync(0xffffffffu, bits & 1u) && lane_id() == 0) set_flag(st, F_NAMES_DIFFER);
        if (__any_sync(0xffffffffu, bits & 2u) && lane_id() == 0) set_err(st, ERR_INVALID);
    }
};

// Name ids of every kernel below 2^24 (per-stream rows with layer classes,
// where the pairing above sees the replayed kernels only).
__global__ void k_check_names24(const uint32_t *__restrict__ name, int64_t n, DevStatus *st) {
    pdl_wait();
    uint32_t acc = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        acc |= name[i];
    if (__any_sync(0xffffffffu, acc >> 24 != 0) && lane_id() == 0) set_err(st, ERR_INVALID);
}

__global__ void k_fill_match(int32_t *out_idx, uint8_t *out_kind, int64_t n) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        out_idx[i] = -1;
        if (out_kind) out_kind[i] = 0;
    }
}

// ------------------------------------------------------------------ general path helpers
// Flags in time order: flag[i] = predicate(korder[i]).
//   what = 0: replayed (layer < 0 or the layer is its class representative)
//   what = 1: layer-tagged (layer >= 0)
__global__ void k_flags(const uint32_t *__restrict__ korder, const int32_t *__restrict__ layer,
                        const int32_t *__restrict__ rep_layer, int64_t n, int what, uint32_t *__restrict__ flag) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int64_t k = korder ? korder[i] : i;
        int32_t l = layer ? layer[k] : -1;
        uint32_t f = what == 0 ? (l < 0 || rep_layer[l] == l) : (l >= 0);
        flag[i] = f;
    }
}
// Compact: list[pos[i]] = korder[i] where flag[i]
__global__ void k_compact(const uint32_t *__restrict__ korder, const uint32_t *__restrict__ flag,
                          const uint32_t *__restrict__ pos, int64_t n, uint32_t *__restrict__ list) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        if (flag[i]) list[pos[i]] = korder ? korder[i] : (uint32_t)i;
}
__global__ void k_gather_u32(const uint32_t *__restrict__ src, const uint32_t *__restrict__ idx, int64_t n,
                             uint32_t *__restrict__ dst) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = idx ? src[idx[i]] : src[i];
}
__global__ void k_gather_i32_as_u32(const int32_t *__restrict__ src, const uint32_t *__restrict__ idx, int64_t n,
                                    uint32_t *__restrict__ dst) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = (uint32_t)src[idx[i]];
}
__global__ void k_max_u32(const uint32_t *__restrict__ a, int64_t n, unsigned long long *out) {
    pdl_wait();
    uint32_t m = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        m = a[i] > m ? a[i] : m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        uint32_t x = __shfl_xor_sync(0xffffffffu, m, o);
        m = x > m ? x : m;
    }
    __shared__ uint32_t sm[32];
    if (lane_id() == 0) sm[threadIdx.x >> 5] = m;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (unsigned w = 1; w < blockDim.x / 32; ++w) m = sm[w] > m ? sm[w] : m;
        if (m) atomicMax(out, (unsigned long long)m);
    }
}
__global__ void k_check_layers(const int32_t *__restrict__ layer, int64_t n, int32_t n_layers,
                               const int32_t *__restrict__ rep_layer, DevStatus *st) {
    pdl_wait();
    unsigned long long rep = 0;
    int bad = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        int32_t l = layer[i];
        if (l < -1 || l >= n_layers) bad = 1;
        else rep += (l < 0 || rep_layer[l] == l);
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
    block_add_u64(rep, &st->cnt[C_REPLAYED], red);
}

__device__ __forceinline__ int64_t lower_bound_u32(const uint32_t *a, int64_t n, uint32_t x) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        int64_t m = (lo + hi) >> 1;
        if (a[m] < x) lo = m + 1; else hi = m;
    }
    return lo;
}
__device__ __forceinline__ int64_t upper_bound_u32(const uint32_t *a, int64_t n, uint32_t x) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        int64_t m = (lo + hi) >> 1;
        if (a[m] <= x) lo = m + 1; else hi = m;
    }
    return lo;
}

// Runs of equal keys in a sorted array.  flag[i] = 1 at each run's first
// element; after an exclusive scan pos[i] counts the runs that start before
// i, so element i lies in run pos[i] + head(i) - 1 and start[pos[i]] = i at
// each head.
__device__ __forceinline__ bool run_head(const uint32_t *a, int64_t i) { return i == 0 || a[i - 1] != a[i]; }

__global__ void k_run_heads(const uint32_t *__restrict__ a, int64_t n, uint32_t *__restrict__ flag) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        flag[i] = run_head(a, i);
}
__global__ void k_run_starts(const uint32_t *__restrict__ a, const uint32_t *__restrict__ pos, int64_t n,
                             uint32_t *__restrict__ start) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        if (run_head(a, i)) start[pos[i]] = (uint32_t)i;
}

// First run r in [0, nr) whose key a[start[r]] is >= x.
__device__ __forceinline__ int64_t lower_bound_runs(const uint32_t *a, const uint32_t *start, int64_t nr, uint32_t x) {
    int64_t lo = 0, hi = nr;
    while (lo < hi) {
        int64_t m = (lo + hi) >> 1;
        if (a[start[m]] < x) lo = m + 1; else hi = m;
    }
    return lo;
}

// Per kernel name run u (replayed kernels sorted by (name, time)): the ncu
// rows of the same name, as the first position b[u] in the sorted rows and
// their count cq[u].  Runs whose kernel and row counts differ are counted
// (and are an error in the error mode).
__global__ void k_run_pair(const uint32_t *__restrict__ skn, const uint32_t *__restrict__ ustart,
                           const uint32_t *__restrict__ n_urun, int64_t nrep, const uint32_t *__restrict__ snn,
                           const uint32_t *__restrict__ vstart, const uint32_t *__restrict__ n_vrun, int64_t M,
                           int mode, uint32_t *__restrict__ b_of, uint32_t *__restrict__ cq_of, DevStatus *st) {
    pdl_wait();
    const int64_t U = *n_urun, V = *n_vrun;
    unsigned long long names_bad = 0;
    for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < U; u += (int64_t)gridDim.x * blockDim.x) {
        const int64_t lo = ustart[u], hi = u + 1 < U ? ustart[u + 1] : nrep;
        const uint32_t name = skn[lo];
        const int64_t v = lower_bound_runs(snn, vstart, V, name);
        const bool found = v < V && snn[vstart[v]] == name;
        const int64_t b = found ? vstart[v] : 0;
        const int64_t cq = found ? (v + 1 < V ? vstart[v + 1] : M) - b : 0;
        b_of[u] = (uint32_t)b;
        cq_of[u] = (uint32_t)cq;
        names_bad += hi - lo != cq;
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, names_bad != 0) && lane_id() == 0 && mode == OPATTR_MISMATCH_ERROR)
        set_err(st, ERR_COUNT);
    block_add_u64(names_bad, &st->cnt[C_NAMES_MISMATCH], red);
}

// Names that have ncu rows but no replayed kernel at all (one thread per
// ncu name run).
__global__ void k_ncu_only_names(const uint32_t *__restrict__ snn, const uint32_t *__restrict__ vstart,
                                 const uint32_t *__restrict__ n_vrun, const uint32_t *__restrict__ skn,
                                 const uint32_t *__restrict__ ustart, const uint32_t *__restrict__ n_urun, int mode,
                                 DevStatus *st) {
    pdl_wait();
    const int64_t U = *n_urun, V = *n_vrun;
    unsigned long long bad = 0;
    for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < V; v += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t name = snn[vstart[v]];
        const int64_t u = lower_bound_runs(skn, ustart, U, name);
        bad += u == U || skn[ustart[u]] != name;
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, bad != 0) && lane_id() == 0 && mode == OPATTR_MISMATCH_ERROR) set_err(st, ERR_COUNT);
    block_add_u64(bad, &st->cnt[C_NAMES_MISMATCH], red);
}

// The ordinal join.  i runs over replayed kernels sorted by (name, time):
//   skn / skj: sorted names, and the time rank j of each (rk[j] = kernel)
//   kpos / ustart / b_of / cq_of: the run tables of skn
//   snj: the row index of each ncu row in name-sorted order
// Kernel i is the o-th of its name with o = i - ustart[run]; its row is the
// o-th row of the name, subject to the mismatch mode.
__global__ void k_ordinal_join(const uint32_t *__restrict__ skn, const uint32_t *__restrict__ skj,
                               const uint32_t *__restrict__ kpos, const uint32_t *__restrict__ ustart,
                               const uint32_t *__restrict__ n_urun, const uint32_t *__restrict__ b_of,
                               const uint32_t *__restrict__ cq_of, const uint32_t *__restrict__ rk, int64_t nrep,
                               const uint32_t *__restrict__ snj, int mode, int32_t *__restrict__ out_idx,
                               uint8_t *__restrict__ out_kind, DevStatus *st) {
    pdl_wait();
    const int64_t U = *n_urun;
    unsigned long long direct = 0, unmatched = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nrep; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t u = (int64_t)kpos[i] + run_head(skn, i) - 1;
        const int64_t lo = ustart[u], hi = u + 1 < U ? ustart[u + 1] : nrep;
        const int64_t cq = cq_of[u], o = i - lo;
        const bool ok = mode == OPATTR_MISMATCH_SKIP_NAME ? (hi - lo == cq) : (o < cq);
        const int32_t idx = ok && o < cq ? (int32_t)snj[b_of[u] + o] : -1;
        const uint32_t k = rk[skj[i]];
        out_idx[k] = idx;
        if (out_kind) out_kind[k] = idx >= 0 ? 1 : 0;
        direct += idx >= 0;
        unmatched += idx < 0;
    }
    __shared__ unsigned long long red[33];
    block_add_u64(direct, &st->cnt[C_DIRECT], red);
    block_add_u64(unmatched, &st->cnt[C_COUNT_UNMATCHED], red);
}

// Broadcast.  i runs over layer-tagged kernels sorted by (layer, time).
//   sll / slj: sorted layer ids and the time rank j of each (lk[j] = kernel)
__global__ void k_dedup_broadcast(const uint32_t *__restrict__ sll, const uint32_t *__restrict__ slj,
                                  const uint32_t *__restrict__ lk, int64_t nl, const int32_t *__restrict__ rep_layer,
                                  const uint32_t *__restrict__ kname, int32_t *__restrict__ out_idx,
                                  uint8_t *__restrict__ out_kind, DevStatus *st) {
    pdl_wait();
    unsigned long long bc = 0, miss = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nl; i += (int64_t)gridDim.x * blockDim.x) {
        uint32_t L = sll[i];
        int32_t rep = rep_layer[L];
        if ((uint32_t)rep == L) continue;                        // the representative itself: replayed
        int64_t lo = (i == 0 || sll[i - 1] != L) ? i : lower_bound_u32(sll, nl, L);
        int64_t p = i - lo;
        int64_t rlo = lower_bound_u32(sll, nl, (uint32_t)rep);
        int64_t rn = upper_bound_u32(sll, nl, (uint32_t)rep) - rlo;
        uint32_t k = lk[slj[i]];
        int32_t idx = -1;
        if (p < rn) {
            uint32_t src = lk[slj[rlo + p]];
            if (kname[src] == kname[k]) idx = out_idx[src];
        }
        out_idx[k] = idx;
        if (out_kind) out_kind[k] = idx >= 0 ? 2 : 0;
        bc += idx >= 0;
        miss += idx < 0;
    }
    __shared__ unsigned long long red[33];
    block_add_u64(bc, &st->cnt[C_BROADCAST], red);
    block_add_u64(miss, &st->cnt[C_DEDUP_MISMATCH], red);
}

// ------------------------------------------------------------------ host
// (name, stream) as one key, name << 8 | stream, for per-stream ordinals; a
// name id of 2^24 or more cannot be packed and is an invalid argument.
__global__ void k_stream_keys(const uint32_t *__restrict__ name, const uint8_t *__restrict__ stream, int64_t n,
                              uint32_t *__restrict__ key, DevStatus *st) {
    pdl_wait();
    int bad = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t x = name[i];
        bad |= x >> 24 != 0;
        key[i] = (x << 8) | stream[i];
    }
    if (bad) set_err(st, ERR_INVALID);
}

__global__ void k_iota(uint32_t *dst, int64_t n) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = (uint32_t)i;
}

static opattr_status read_u64(Ctx &c, const unsigned long long *d, unsigned long long *h) {
    if (cudaMemcpyAsync(h, d, sizeof(*h), cudaMemcpyDeviceToHost, c.stream) != cudaSuccess ||
        cudaStreamSynchronize(c.stream) != cudaSuccess)
        return cuda_status(c, cudaGetLastError());
    return OPATTR_OK;
}

// The stream-partitioned pairing over n replayed kernels (list rk, or the
// kernel array itself when rk is null) and the n rows.  Scratch: nb (n
// bytes), nv0 / nv1 (n).
static void stream_pairs(Ctx &c, const opattr_kernels *kern, const opattr_ncu *ncu, const uint32_t *rk, int64_t n,
                         uint8_t *nb, uint32_t *nv0, uint32_t *nv1, uint32_t *hist, uint32_t *part, int32_t *out_idx,
                         uint8_t *out_kind) {
    // rows: one 8-bit radix pass (it only reads the row streams)
    uint8_t *ko;
    uint32_t *pn;
    radix_sort_pairs<uint8_t>(c, const_cast<uint8_t *>(ncu->stream), nv0, nb, nv1, n, 8, true, hist, part, &ko, &pn);
    // kernels: ranked by stream, each paired in the same pass
    const StreamDigit dg{rk, kern->stream};
    const uint32_t *offs = digit_offsets(c, dg, n, hist, part);
    const StreamPairs ep{rk, pn, kern->name_id, ncu->name_id, kern->stream, ncu->stream, out_idx, out_kind,
                         c.d_status};
    digit_rank(c, "match_stream_pairs", dg, n, offs, ep);
}

opattr_status do_match(Ctx &c, const opattr_kernels *kern, const opattr_ncu *ncu, const opattr_dedup *dd,
                       int32_t *out_idx, uint8_t *out_kind, opattr_match_summary *sum) {
    const int64_t K = kern->n, M = ncu->n;
    c.rows_identity = false;
    if (K < 0 || M < 0 || K >= (1ll << 31) || M >= (1ll << 31)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->stream || !kern->start_ns || !kern->name_id || !out_idx)) return OPATTR_E_INVALID_ARG;
    if (M > 0 && !ncu->name_id) return OPATTR_E_INVALID_ARG;
    const int mode = (int)c.cfg.mismatch;
    const bool dedup_on = c.cfg.dedup && dd && kern->layer_id;
    std::vector<int32_t> rep_layer;
    if (dedup_on) {
        if (dd->n_layers < 0 || dd->n_classes < 0 || (dd->n_layers > 0 && !dd->class_of_layer) ||
            (dd->n_classes > 0 && !dd->rep_of_class))
            return OPATTR_E_INVALID_ARG;
        for (int32_t l = 0; l < dd->n_layers; ++l)
            if (dd->class_of_layer[l] < 0 || dd->class_of_layer[l] >= dd->n_classes) return OPATTR_E_INVALID_ARG;
        for (int32_t q = 0; q < dd->n_classes; ++q) {
            int32_t r = dd->rep_of_class[q];
            if (r < 0 || r >= dd->n_layers || dd->class_of_layer[r] != q) return OPATTR_E_INVALID_ARG;
        }
        rep_layer.resize(dd->n_layers > 0 ? dd->n_layers : 1);
        for (int32_t l = 0; l < dd->n_layers; ++l) rep_layer[l] = dd->rep_of_class[dd->class_of_layer[l]];
    }
    const int64_t NL = dedup_on ? (dd->n_layers > 0 ? dd->n_layers : 1) : 1;
    const int64_t NX = std::max(K, M);
    const bool per_stream = ncu->stream != nullptr;
    if (per_stream && M > 0 && !ncu->name_id) return OPATTR_E_INVALID_ARG;
    // within a join the identity pairing ran beside the enclosure: with the
    // kernels in time order (the enclosure's verdict) and every name equal,
    // its outputs are the match
    // (with the enclosure's status still to be read, the names are taken to
    // agree; the join checks that verdict with the aggregation's status)
    if (c.spec_ran && c.order_from_enclose && c.enclose_k_sorted == 1 && c.spec_kname == kern->name_id &&
        c.spec_nname == ncu->name_id && c.spec_idx == out_idx &&
        c.spec_kind == out_kind && c.spec_k == K && K == M && !dedup_on && !per_stream &&
        (c.enclose_pending || !(c.h_status->flags & F_NAMES_DIFFER))) {
        opattr_match_summary S{};
        S.kernels = K;
        S.replayed = K;
        S.direct = K;
        S.fast_path = 1;
        if (sum) *sum = S;
        c.rows_identity = true;
        return OPATTR_OK;
    }
    Need nd;
    if (per_stream) nd.add<uint32_t>(K).add<uint32_t>(M);        // (name, stream) keys
    nd.add<int32_t>(NL);
    for (int i = 0; i < 5; ++i) nd.add<uint32_t>(K);                 // flag, pos, rk, lk, keys
    for (int i = 0; i < 3; ++i) nd.add<uint32_t>(NX);                // sort buffers
    for (int i = 0; i < 4; ++i) nd.add<uint32_t>(M);                 // ncu sort
    nd.add<uint32_t>(radix_hist_elems(NX)).add<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(NX), NX)));
    nd.add<unsigned long long>(4);
    size_t need = nd.bytes + kernel_order_scratch(K) + 4096;
    opattr_status st = ensure_arena(c, need);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;
    int32_t *d_rep = a.take<int32_t>(NL);
    uint32_t *flag = a.take<uint32_t>(K), *pos = a.take<uint32_t>(K), *rk = a.take<uint32_t>(K);
    uint32_t *lk = a.take<uint32_t>(K), *k0 = a.take<uint32_t>(K);
    uint32_t *s0 = a.take<uint32_t>(NX), *s1 = a.take<uint32_t>(NX), *s2 = a.take<uint32_t>(NX);
    uint32_t *n0 = a.take<uint32_t>(M), *n1 = a.take<uint32_t>(M), *n2 = a.take<uint32_t>(M), *n3 = a.take<uint32_t>(M);
    uint32_t *hist = a.take<uint32_t>(radix_hist_elems(NX));
    uint32_t *part = a.take<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(NX), NX)));
    unsigned long long *dsm = a.take<unsigned long long>(4);
    if (!d_rep || !flag || !pos || !rk || !lk || !k0 || !s0 || !s1 || !s2 || !n0 || !n1 || !n2 || !n3 || !hist ||
        !part || !dsm)
        return OPATTR_E_OOM;
    if (dedup_on && dd->n_layers > 0)
        cudaMemcpyAsync(d_rep, rep_layer.data(), sizeof(int32_t) * dd->n_layers, cudaMemcpyHostToDevice, c.stream);
    // the matching key: the name id, or (name, stream) when the rows carry
    // streams (built only if the general path runs)
    const uint32_t *kname = kern->name_id, *nname = ncu->name_id;
    uint32_t *kkey = nullptr, *nkey = nullptr;
    if (per_stream) {
        kkey = a.take<uint32_t>(K);
        nkey = a.take<uint32_t>(M);
        if ((K > 0 && !kkey) || (M > 0 && !nkey)) return OPATTR_E_OOM;
    }

    const unsigned gK = grid_for(K, 256, REDUCE_GRID);
    // within a join the enclosure has just verified these records' order, and
    // kept their time order when they were out of it
    const bool known_sorted = c.order_from_enclose && c.enclose_k_sorted == 1;
    const bool known_unsorted = c.order_from_enclose && c.enclose_k_sorted == 0 && c.join_korder;
    if (!known_sorted && !known_unsorted) check_kernel_order(c, kern->stream, kern->start_ns, K);
    if (dedup_on && K > 0)
        launch(c, "check_layers", k_check_layers, dim3(gK), dim3(256), 0, kern->layer_id, K, dd->n_layers,
               (const int32_t *)d_rep, c.d_status);
    if (per_stream && dedup_on && K > 0)
        launch(c, "check_names24", k_check_names24, dim3(grid_for(K, 256 * 8, REDUCE_GRID)), dim3(256), 0,
               kern->name_id, K, c.d_status);
    // Speculative fast paths, taking the kernel array to be in time order
    // (confirmed or refuted by the order check in the same batch).
    const bool try_identity = !dedup_on && !per_stream && K == M && K > 0 && !known_unsorted;
    const bool try_streams = !dedup_on && per_stream && K == M && K > 0 && !known_unsorted;
    if (try_identity)
        launch(c, "match_identity", k_match_identity, dim3(grid_for(K, 256 * 16, REDUCE_GRID)), dim3(256), 0,
               kname, nname, K, out_idx, out_kind, identity_vec(kname, nname, out_idx, out_kind), c.d_status);
    if (try_streams)
        stream_pairs(c, kern, ncu, nullptr, K, reinterpret_cast<uint8_t *>(n2), n0, n1, hist, part, out_idx,
                     out_kind);
    if ((st = read_status(c))) return st;
    if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    const bool k_sorted = known_sorted || (!known_unsorted && !(c.h_status->flags & F_K_UNSORTED));
    opattr_match_summary S{};
    S.kernels = K;
    S.replayed = dedup_on ? (int64_t)c.h_status->cnt[C_REPLAYED] : K;
    if ((try_identity || try_streams) && k_sorted && !(c.h_status->flags & F_NAMES_DIFFER)) {
        S.direct = K;
        S.fast_path = 1;
        if (sum) *sum = S;
        return OPATTR_OK;
    }
    // the speculative verdicts are spent: later checks start from clear flags
    cudaMemsetAsync(&c.d_status->flags, 0, sizeof(unsigned), c.stream);

    // ---- general path
    if (K > 0) launch(c, "fill_match", k_fill_match, dim3(gK), dim3(256), 0, out_idx, out_kind, K);
    uint32_t *korder = nullptr;
    if (!k_sorted && K > 0) {
        korder = known_unsorted ? c.join_korder : kernel_time_order(c, a, kern->stream, kern->start_ns, K);
        if (!korder) return OPATTR_E_OOM;
    }
    // rk[j] = kernel index of the j-th replayed kernel in time order
    int64_t nrep = K;
    if (dedup_on && K > 0) {
        launch(c, "flags", k_flags, dim3(gK), dim3(256), 0, (const uint32_t *)korder, kern->layer_id,
               (const int32_t *)d_rep, K, 0, flag);
        scan_exclusive_u32(c, flag, pos, K, part, nullptr);
        launch(c, "compact", k_compact, dim3(gK), dim3(256), 0, (const uint32_t *)korder, (const uint32_t *)flag,
               (const uint32_t *)pos, K, rk);
        nrep = S.replayed;
    } else if (K > 0) {
        if (korder) cudaMemcpyAsync(rk, korder, sizeof(uint32_t) * K, cudaMemcpyDeviceToDevice, c.stream);
        else launch(c, "iota", k_iota, dim3(gK), dim3(256), 0, rk, K);
    }
    bool direct_done = false;
    // rows equal to the replayed kernels in time order, tried before the name
    // sorts: with layer deduplication, or when the kernels were out of time order
    const bool retry_streams = per_stream && (dedup_on || korder) && nrep == M && nrep > 0;
    if (((dedup_on || korder) && !per_stream && nrep == M && nrep > 0) || retry_streams) {
        if (retry_streams)
            stream_pairs(c, kern, ncu, rk, nrep, reinterpret_cast<uint8_t *>(n2), n0, n1, hist, part, out_idx,
                         out_kind);
        else
            launch(c, "match_identity_list", k_match_identity_list, dim3(grid_for(nrep, 256, REDUCE_GRID)),
                   dim3(256), 0, (const uint32_t *)rk, kname, nname, nrep, out_idx, out_kind, c.d_status);
        if ((st = read_status(c))) return st;
        if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
        direct_done = !(c.h_status->flags & F_NAMES_DIFFER);
        if (direct_done) S.fast_path = 1;
        else launch(c, "fill_match", k_fill_match, dim3(gK), dim3(256), 0, out_idx, out_kind, K);
    }
    if (!direct_done && (nrep > 0 || M > 0)) {
        if (per_stream) {
            if (K > 0)
                launch(c, "stream_keys", k_stream_keys, dim3(grid_for(K, 256, REDUCE_GRID)), dim3(256), 0,
                       kern->name_id, kern->stream, K, kkey, c.d_status);
            if (M > 0)
                launch(c, "stream_keys", k_stream_keys, dim3(grid_for(M, 256, REDUCE_GRID)), dim3(256), 0,
                       ncu->name_id, ncu->stream, M, nkey, c.d_status);
            kname = kkey;
            nname = nkey;
        }
        cudaMemsetAsync(dsm, 0, sizeof(unsigned long long), c.stream);
        if (nrep > 0) {
            launch(c, "gather_names", k_gather_u32, dim3(grid_for(nrep, 256, REDUCE_GRID)), dim3(256), 0, kname,
                   (const uint32_t *)rk, nrep, k0);
            launch(c, "max_name", k_max_u32, dim3(grid_for(nrep, 256, 4096)), dim3(256), 0, (const uint32_t *)k0, nrep,
                   dsm);
        }
        if (M > 0) {
            cudaMemcpyAsync(n0, nname, sizeof(uint32_t) * M, cudaMemcpyDeviceToDevice, c.stream);
            launch(c, "max_name", k_max_u32, dim3(grid_for(M, 256, 4096)), dim3(256), 0, (const uint32_t *)n0, M, dsm);
        }
        unsigned long long hmax = 0;
        if ((st = read_u64(c, dsm, &hmax))) return st;
        const int bits = bits_for(hmax);
        uint32_t *skn = nullptr, *skj = nullptr, *snn = n0, *snj = n1;
        if (nrep > 0) radix_sort_pairs<uint32_t>(c, k0, s0, s1, s2, nrep, bits, true, hist, part, &skn, &skj);
        if (M > 0) radix_sort_pairs<uint32_t>(c, n0, n1, n2, n3, M, bits, true, hist, part, &snn, &snj);
        // run tables of both sorted name arrays (pos / start pairs in the
        // buffers the sorts left free)
        uint32_t *kfree0 = skn == k0 ? s1 : k0, *kfree1 = skn == k0 ? s2 : s0;
        uint32_t *nfree0 = snn == n0 ? n2 : n0, *nfree1 = snn == n0 ? n3 : n1;
        uint32_t *kpos = flag, *ustart = pos, *b_of = kfree0, *cq_of = kfree1, *vpos = nfree0, *vstart = nfree1;
        uint32_t *n_urun = reinterpret_cast<uint32_t *>(dsm + 2), *n_vrun = reinterpret_cast<uint32_t *>(dsm + 3);
        if (nrep > 0) {
            launch(c, "run_heads", k_run_heads, dim3(grid_for(nrep, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)skn, nrep, kpos);
        }
        scan_exclusive_u32(c, kpos, kpos, nrep, part, n_urun);
        if (nrep > 0)
            launch(c, "run_starts", k_run_starts, dim3(grid_for(nrep, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)skn, (const uint32_t *)kpos, nrep, ustart);
        if (M > 0)
            launch(c, "run_heads", k_run_heads, dim3(grid_for(M, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)snn, M, vpos);
        scan_exclusive_u32(c, vpos, vpos, M, part, n_vrun);
        if (M > 0)
            launch(c, "run_starts", k_run_starts, dim3(grid_for(M, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)snn, (const uint32_t *)vpos, M, vstart);
        if (nrep > 0) {
            launch(c, "run_pair", k_run_pair, dim3(grid_for(nrep, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)skn, (const uint32_t *)ustart, (const uint32_t *)n_urun, nrep,
                   (const uint32_t *)snn, (const uint32_t *)vstart, (const uint32_t *)n_vrun, M, mode, b_of, cq_of,
                   c.d_status);
            launch(c, "ordinal_join", k_ordinal_join, dim3(grid_for(nrep, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)skn, (const uint32_t *)skj, (const uint32_t *)kpos, (const uint32_t *)ustart,
                   (const uint32_t *)n_urun, (const uint32_t *)b_of, (const uint32_t *)cq_of, (const uint32_t *)rk,
                   nrep, (const uint32_t *)snj, mode, out_idx, out_kind, c.d_status);
        }
        if (M > 0)
            launch(c, "ncu_only_names", k_ncu_only_names, dim3(grid_for(M, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)snn, (const uint32_t *)vstart, (const uint32_t *)n_vrun, (const uint32_t *)skn,
                   (const uint32_t *)ustart, (const uint32_t *)n_urun, mode, c.d_status);
    }
    if (dedup_on && K > 0) {
        // positions within layers: layer-tagged kernels in time order, sorted by layer
        launch(c, "flags", k_flags, dim3(gK), dim3(256), 0, (const uint32_t *)korder, kern->layer_id,
               (const int32_t *)d_rep, K, 1, flag);
        uint32_t *ntag = reinterpret_cast<uint32_t *>(dsm + 1);
        scan_exclusive_u32(c, flag, pos, K, part, ntag);
        launch(c, "compact", k_compact, dim3(gK), dim3(256), 0, (const uint32_t *)korder, (const uint32_t *)flag,
               (const uint32_t *)pos, K, lk);
        unsigned long long ntag_h = 0;
        if ((st = read_u64(c, dsm + 1, &ntag_h))) return st;
        const int64_t nlk = (int64_t)(ntag_h & 0xFFFFFFFFull);
        if (nlk > 0) {
            launch(c, "gather_layers", k_gather_i32_as_u32, dim3(grid_for(nlk, 256, REDUCE_GRID)), dim3(256), 0,
                   kern->layer_id, (const uint32_t *)lk, nlk, k0);
            uint32_t *sll, *slj;
            radix_sort_pairs<uint32_t>(c, k0, s0, s1, s2, nlk,
                                       bits_for((uint64_t)(dd->n_layers > 0 ? dd->n_layers - 1 : 0)), true, hist, part,
                                       &sll, &slj);
            launch(c, "dedup_broadcast", k_dedup_broadcast, dim3(grid_for(nlk, 256, REDUCE_GRID)), dim3(256), 0,
                   (const uint32_t *)sll, (const uint32_t *)slj, (const uint32_t *)lk, nlk, (const int32_t *)d_rep,
                   kern->name_id, out_idx, out_kind, c.d_status);   // plain names: a class may span streams
        }
    }
    if ((st = read_status(c))) return st;
    const DevStatus &H = *c.h_status;
    if (H.err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    if (H.err & ERR_COUNT) return OPATTR_E_COUNT_MISMATCH;
    S.direct = direct_done ? nrep : (int64_t)H.cnt[C_DIRECT];
    S.broadcast = (int64_t)H.cnt[C_BROADCAST];
    S.names_mismatched = (int64_t)H.cnt[C_NAMES_MISMATCH];
    S.count_unmatched = direct_done ? 0 : (int64_t)H.cnt[C_COUNT_UNMATCHED];
    S.dedup_mismatch = (int64_t)H.cnt[C_DEDUP_MISMATCH];
    S.unmatched = K - S.direct - S.broadcast;
    if (sum) *sum = S;
    if (mode == OPATTR_MISMATCH_SKIP_NAME && S.names_mismatched > 0) return OPATTR_W_COUNT_MISMATCH;
    if (mode == OPATTR_MISMATCH_PREFIX && S.count_unmatched > 0) return OPATTR_W_COUNT_MISMATCH;
    if (S.dedup_mismatch > 0) return OPATTR_W_DEDUP_MISMATCH;
    return OPATTR_OK;
}

}  // namespace opattr
