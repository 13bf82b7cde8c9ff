// attribute.cu -- the attribution tiers of Fig. 2 on the GPU: torch.profiler
// correlation (HIGH, Sec. 3.4), NVTX enclosure (Sec. 3.5) and the Inductor
// fusion map (Sec. 3.6).
//
// Invocation indices.  The HIGH tier is keyed by (kernel name, invocation
// index), the index being the kernel's rank among all kernels of its name in
// time order.  A stable radix sort of the kernels' name ids, taken in time
// order, puts each name's launches in one run in launch order, so the kernel
// at sorted position i has index i - start of its run.  The correlation map
// is scattered into a table over sorted positions: the entry (name, inv, op)
// lands at start(run of name) + inv when the name has a run longer than inv;
// a second entry landing on an occupied slot is a repeated pair.  Reading the
// table at each kernel's sorted position gives its HIGH operator, with no
// per-kernel search.
//
// Tiers.  One pass over the kernels then takes the first tier with an
// operator (HIGH, then the enclosing range's operator, then the fusion map's
// operator for the kernel's name) and records the fusion enrichment.
#include <algorithm>

#include "sort.cuh"
#include "util.cuh"

namespace opattr {

// ------------------------------------------------------------------ checks
// Range index in [-1, R) and, when a range is given, an operator below n_ops;
// the largest name id (radix sort width).
__global__ void k_attr_check_kernels(const int32_t *__restrict__ rok, const uint32_t *__restrict__ r_op, int64_t R,
                                     const uint32_t *__restrict__ name, int64_t K, uint32_t n_ops,
                                     unsigned long long *max_name, DevStatus *st) {
    pdl_wait();
    int bad = 0;
    uint32_t mx = 0;
    for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < K; k += (int64_t)gridDim.x * blockDim.x) {
        const int32_t r = rok[k];
        if (r < -1 || r >= R) bad = 1;
        else if (r >= 0 && r_op[r] >= n_ops) bad = 1;
        const uint32_t x = name[k];
        mx = x > mx ? x : mx;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const uint32_t y = __shfl_xor_sync(0xffffffffu, mx, o);
        mx = y > mx ? y : mx;
    }
    if (lane_id() == 0 && mx) atomicMax(max_name, (unsigned long long)mx);
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
}

// Every operator of a table below n_ops (OPATTR_OP_NONE allowed where `none_ok`).
__global__ void k_attr_check_ops(const uint32_t *__restrict__ op, int64_t n, uint32_t n_ops, int none_ok,
                                 DevStatus *st) {
    pdl_wait();
    int bad = 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t x = op[i];
        bad |= x >= n_ops && !(none_ok && x == OPATTR_OP_NONE);
    }
    if (__any_sync(0xffffffffu, bad) && lane_id() == 0) set_err(st, ERR_INVALID);
}

// ------------------------------------------------------------------ HIGH tier
__global__ void k_gather_names(const uint32_t *__restrict__ name, const uint32_t *__restrict__ korder, int64_t n,
                               uint32_t *__restrict__ dst) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        dst[i] = name[korder ? korder[i] : i];
}
__device__ __forceinline__ bool run_head_u32(const uint32_t *a, int64_t i) { return i == 0 || a[i - 1] != a[i]; }

__global__ void k_attr_heads(const uint32_t *__restrict__ skn, int64_t n, uint32_t *__restrict__ flag) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        flag[i] = run_head_u32(skn, i);
}
__global__ void k_attr_starts(const uint32_t *__restrict__ skn, const uint32_t *__restrict__ pos, int64_t n,
                              uint32_t *__restrict__ start) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        if (run_head_u32(skn, i)) start[pos[i]] = (uint32_t)i;
}

// Each correlation entry to its slot: the sorted position of the launch it
// names.  Slots start as OPATTR_OP_NONE; an occupied slot means the pair was
// repeated.
__global__ void k_corr_scatter(const uint32_t *__restrict__ c_name, const uint32_t *__restrict__ c_inv,
                               const uint32_t *__restrict__ c_op, int64_t nc, const uint32_t *__restrict__ skn,
                               const uint32_t *__restrict__ ustart, const uint32_t *__restrict__ n_urun, int64_t K,
                               uint32_t *__restrict__ table, DevStatus *st) {
    pdl_wait();
    const int64_t U = *n_urun;
    unsigned long long used = 0;
    int dup = 0;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nc; e += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t name = c_name[e];
        int64_t lo = 0, hi = U;                   // first run whose name is >= name
        while (lo < hi) {
            const int64_t m = (lo + hi) >> 1;
            if (skn[ustart[m]] < name) lo = m + 1; else hi = m;
        }
        if (lo == U || skn[ustart[lo]] != name) continue;
        const int64_t s = ustart[lo], len = (lo + 1 < U ? (int64_t)ustart[lo + 1] : K) - s;
        const uint32_t inv = c_inv[e];
        if ((int64_t)inv >= len) continue;
        const uint32_t old = atomicExch(&table[s + inv], c_op[e]);
        dup |= old != OPATTR_OP_NONE;
        used++;
    }
    __shared__ unsigned long long red[33];
    if (__any_sync(0xffffffffu, dup) && lane_id() == 0) set_err(st, ERR_INVALID);
    block_add_u64(used, &st->cnt[C_CORR_USED], red);
}

// The HIGH operator of each kernel: the table at its sorted position.
__global__ void k_corr_gather(const uint32_t *__restrict__ table, const uint32_t *__restrict__ skj,
                              const uint32_t *__restrict__ korder, int64_t K, uint32_t *__restrict__ hi_op) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < K; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t j = skj[i];
        hi_op[korder ? korder[j] : j] = table[i];
    }
}

// ------------------------------------------------------------------ tiers
struct TierIn {
    const int32_t *rok;
    const uint32_t *r_op;
    const uint32_t *name;
    const uint8_t *nop;          // n_op_enclosing, or NULL
    const uint32_t *hi_op;       // HIGH operator per kernel, or NULL
    const uint32_t *f_op;        // fusion operator per name, or NULL
    const uint8_t *f_len;        // fused list length per name, or NULL (1)
    int64_t n_names;
    int64_t K;
    uint32_t *op_of_kernel;
    uint8_t *tier;
    uint32_t *fused_with;
    uint8_t *is_fused;
};

__global__ void k_tiers(TierIn A, DevStatus *st) {
    pdl_wait();
    constexpr int U = 4;                      // kernels per thread per round, loads issued together
    unsigned long long n_high = 0, n_nvtx = 0, n_ind = 0, n_fused = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t k0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k0 - threadIdx.x < A.K; k0 += stride * U) {
        uint32_t oh[U], nm[U], rop[U], of[U];
        int32_t r[U];
        unsigned flen[U], nk[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {             // lane-consecutive kernels: coalesced
            const int64_t k = k0 + u * stride;
            const bool in = k < A.K;
            oh[u] = in && A.hi_op ? A.hi_op[k] : OPATTR_OP_NONE;
            r[u] = in ? A.rok[k] : -1;
            nm[u] = in ? A.name[k] : 0u;
            nk[u] = in && A.nop ? A.nop[k] : 0u;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {             // dependent gathers, also together
            const bool has_f = A.f_op && (int64_t)nm[u] < A.n_names && k0 + u * stride < A.K;
            rop[u] = r[u] >= 0 ? A.r_op[r[u]] : OPATTR_OP_NONE;
            of[u] = has_f ? A.f_op[nm[u]] : OPATTR_OP_NONE;
            flen[u] = has_f && A.f_len ? A.f_len[nm[u]] : 1u;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t k = k0 + u * stride;
            if (k >= A.K) break;
            uint32_t op = OPATTR_OP_NONE;
            uint8_t t = OPATTR_TIER_NONE;
            if (oh[u] != OPATTR_OP_NONE) {
                op = oh[u];
                t = OPATTR_TIER_HIGH;
            } else if (r[u] >= 0) {
                op = rop[u];
                t = OPATTR_TIER_NVTX;
            } else if (of[u] != OPATTR_OP_NONE) {
                op = of[u];
                t = OPATTR_TIER_INDUCTOR;
            }
            const bool fused = (of[u] != OPATTR_OP_NONE && flen[u] > 1) || (t == OPATTR_TIER_NVTX && nk[u] > 1);
            A.op_of_kernel[k] = op;
            if (A.tier) A.tier[k] = t;
            if (A.fused_with) A.fused_with[k] = of[u];
            if (A.is_fused) A.is_fused[k] = fused ? 1 : 0;
            n_high += t == OPATTR_TIER_HIGH;
            n_nvtx += t == OPATTR_TIER_NVTX;
            n_ind += t == OPATTR_TIER_INDUCTOR;
            n_fused += fused;
        }
    }
    __shared__ unsigned long long red[33];
    block_add_u64(n_high, &st->cnt[C_TIER_HIGH], red);
    block_add_u64(n_nvtx, &st->cnt[C_TIER_NVTX], red);
    block_add_u64(n_ind, &st->cnt[C_TIER_INDUCTOR], red);
    block_add_u64(n_fused, &st->cnt[C_FUSED], red);
}

// ------------------------------------------------------------------ host
static opattr_status read_u64(Ctx &c, const unsigned long long *d, unsigned long long *h) {
    if (cudaMemcpyAsync(h, d, sizeof(*h), cudaMemcpyDeviceToHost, c.stream) != cudaSuccess ||
        cudaStreamSynchronize(c.stream) != cudaSuccess)
        return cuda_status(c, cudaGetLastError());
    return OPATTR_OK;
}

opattr_status do_attribute(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                           const uint8_t *nop, const opattr_corr *corr, const opattr_fusion *fusion,
                           uint32_t n_ops, uint32_t *op_of_kernel, uint8_t *tier, uint32_t *fused_with,
                           uint8_t *is_fused, opattr_attr_summary *sum) {
    const int64_t K = kern->n, R = rng->n;
    const int64_t NC = corr ? corr->n : 0, NF = fusion ? fusion->n_names : 0;
    if (K < 0 || R < 0 || NC < 0 || NF < 0 || K >= (1ll << 31)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && (!kern->name_id || !rok || !op_of_kernel)) return OPATTR_E_INVALID_ARG;
    if (K > 0 && NC > 0 && (!kern->stream || !kern->start_ns)) return OPATTR_E_INVALID_ARG;
    if (R > 0 && !rng->op_id) return OPATTR_E_INVALID_ARG;
    if (NC > 0 && (!corr->name_id || !corr->invocation || !corr->op_id)) return OPATTR_E_INVALID_ARG;
    if (NF > 0 && !fusion->op_of_name) return OPATTR_E_INVALID_ARG;
    const bool high = NC > 0 && K > 0;

    Need nd;
    nd.add<unsigned long long>(4);
    if (high) {
        for (int i = 0; i < 8; ++i) nd.add<uint32_t>(K);    // names, sort x3, flag/pos, starts, table, hi_op
        nd.add<uint32_t>(radix_hist_elems(K)).add<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), K)));
        nd.bytes += kernel_order_scratch(K);
    }
    opattr_status st = ensure_arena(c, nd.bytes + 4096);
    if (st) return st;
    Arena a(c);
    if ((st = reset_status(c))) return st;
    unsigned long long *dsm = a.take<unsigned long long>(4);
    if (!dsm) return OPATTR_E_OOM;
    cudaMemsetAsync(dsm, 0, 4 * sizeof(unsigned long long), c.stream);

    const unsigned gK = grid_for(K, 256, REDUCE_GRID);
    if (K > 0)
        launch(c, "attr_check", k_attr_check_kernels, dim3(gK), dim3(256), 0, rok, rng->op_id, R, kern->name_id, K,
               n_ops, dsm, c.d_status);
    if (NC > 0)
        launch(c, "attr_check_ops", k_attr_check_ops, dim3(grid_for(NC, 256, REDUCE_GRID)), dim3(256), 0,
               corr->op_id, NC, n_ops, 0, c.d_status);
    if (NF > 0)
        launch(c, "attr_check_ops", k_attr_check_ops, dim3(grid_for(NF, 256, REDUCE_GRID)), dim3(256), 0,
               fusion->op_of_name, NF, n_ops, 1, c.d_status);
    if (high) check_kernel_order(c, kern->stream, kern->start_ns, K);
    if ((st = read_status(c))) return st;
    if (c.h_status->err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    const bool k_sorted = !(c.h_status->flags & F_K_UNSORTED);

    uint32_t *hi_op = nullptr;
    if (high) {
        unsigned long long hmax = 0;
        if ((st = read_u64(c, dsm, &hmax))) return st;
        uint32_t *k0 = a.take<uint32_t>(K), *s0 = a.take<uint32_t>(K), *s1 = a.take<uint32_t>(K);
        uint32_t *s2 = a.take<uint32_t>(K), *pos = a.take<uint32_t>(K), *ustart = a.take<uint32_t>(K);
        uint32_t *table = a.take<uint32_t>(K);
        hi_op = a.take<uint32_t>(K);
        uint32_t *hist = a.take<uint32_t>(radix_hist_elems(K));
        uint32_t *part = a.take<uint32_t>(scan_scratch_elems(std::max(radix_hist_elems(K), K)));
        if (!k0 || !s0 || !s1 || !s2 || !pos || !ustart || !table || !hi_op || !hist || !part) return OPATTR_E_OOM;
        uint32_t *korder = nullptr;
        if (!k_sorted) {
            korder = kernel_time_order(c, a, kern->stream, kern->start_ns, K);
            if (!korder) return OPATTR_E_OOM;
        }
        // names in time order, sorted stably: each name's launches in one run
        launch(c, "attr_names", k_gather_names, dim3(gK), dim3(256), 0, kern->name_id, (const uint32_t *)korder, K,
               k0);
        uint32_t *skn, *skj;
        radix_sort_pairs<uint32_t>(c, k0, s0, s1, s2, K, bits_for(hmax), true, hist, part, &skn, &skj);
        uint32_t *n_urun = reinterpret_cast<uint32_t *>(dsm + 1);
        launch(c, "attr_heads", k_attr_heads, dim3(gK), dim3(256), 0, (const uint32_t *)skn, K, pos);
        scan_exclusive_u32(c, pos, pos, K, part, n_urun);
        launch(c, "attr_starts", k_attr_starts, dim3(gK), dim3(256), 0, (const uint32_t *)skn, (const uint32_t *)pos,
               K, ustart);
        cudaMemsetAsync(table, 0xFF, sizeof(uint32_t) * K, c.stream);
        launch(c, "corr_scatter", k_corr_scatter, dim3(grid_for(NC, 256, REDUCE_GRID)), dim3(256), 0,
               corr->name_id, corr->invocation, corr->op_id, NC, (const uint32_t *)skn, (const uint32_t *)ustart,
               (const uint32_t *)n_urun, K, table, c.d_status);
        launch(c, "corr_gather", k_corr_gather, dim3(gK), dim3(256), 0, (const uint32_t *)table,
               (const uint32_t *)skj, (const uint32_t *)korder, K, hi_op);
    }
    if (K > 0) {
        TierIn A;
        A.rok = rok;
        A.r_op = rng->op_id;
        A.name = kern->name_id;
        A.nop = nop;
        A.hi_op = hi_op;
        A.f_op = NF > 0 ? fusion->op_of_name : nullptr;
        A.f_len = NF > 0 ? fusion->list_len : nullptr;
        A.n_names = NF;
        A.K = K;
        A.op_of_kernel = op_of_kernel;
        A.tier = tier;
        A.fused_with = fused_with;
        A.is_fused = is_fused;
        launch(c, "tiers", k_tiers, dim3(grid_for(K, 256 * 4, REDUCE_GRID)), dim3(256), 0, A, c.d_status);
    }
    if ((st = read_status(c))) return st;
    const DevStatus &H = *c.h_status;
    if (H.err & ERR_INVALID) return OPATTR_E_INVALID_ARG;
    if (sum) {
        opattr_attr_summary S{};
        S.kernels = K;
        S.high = (int64_t)H.cnt[C_TIER_HIGH];
        S.nvtx = (int64_t)H.cnt[C_TIER_NVTX];
        S.inductor = (int64_t)H.cnt[C_TIER_INDUCTOR];
        S.none = K - S.high - S.nvtx - S.inductor;
        S.fused = (int64_t)H.cnt[C_FUSED];
        S.corr_used = (int64_t)H.cnt[C_CORR_USED];
        *sum = S;
    }
    return OPATTR_OK;
}

}  // namespace opattr
