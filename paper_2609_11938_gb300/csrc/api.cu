// api.cu -- the C ABI of libopattr: context life cycle, scratch arena, status
// block, launch timing, and the calls of the join.
#include <nvtx3/nvToolsExt.h>
#include <stdlib.h>

#include <algorithm>
#include <new>

#include "common.cuh"

// One NVTX range per call of the C ABI, named after the entry point, so a
// timeline (Nsight Systems) shows the library's calls around their kernels.
// Header-only NVTX: without a tool attached a push or pop costs a few
// nanoseconds.
struct NvtxCall {
    explicit NvtxCall(const char *name) { nvtxRangePushA(name); }
    ~NvtxCall() { nvtxRangePop(); }
    NvtxCall(const NvtxCall &) = delete;
    NvtxCall &operator=(const NvtxCall &) = delete;
};

namespace opattr {

opattr_status do_enclose(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, int32_t *out_range,
                         uint8_t *out_nop);
opattr_status do_match(Ctx &c, const opattr_kernels *kern, const opattr_ncu *ncu, const opattr_dedup *dd,
                       int32_t *out_idx, uint8_t *out_kind, opattr_match_summary *sum);
opattr_status do_aggregate(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                           const opattr_ncu *ncu, const int32_t *nidx, uint32_t n_ops,
                           const opattr_op_aggregates *out, opattr_totals *tot_out);

opattr_status do_attribute(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                           const uint8_t *nop, const opattr_corr *corr, const opattr_fusion *fusion,
                           uint32_t n_ops, uint32_t *op_of_kernel, uint8_t *tier, uint32_t *fused_with,
                           uint8_t *is_fused, opattr_attr_summary *sum);

opattr_status do_rollup(Ctx &c, const opattr_kernels *kern, const opattr_ranges *rng, const int32_t *rok,
                        const opattr_ncu *ncu, const int32_t *nidx, uint32_t n_ops, const uint32_t *class_of_op,
                        uint32_t n_classes, const opattr_op_aggregates *out);

opattr_status cuda_status(Ctx &c, cudaError_t e) {
    if (e == cudaSuccess) e = c.last_error;
    if (e == cudaSuccess) return OPATTR_OK;
    c.last_error = e;
    c.broken = true;
    return OPATTR_E_CUDA;
}

// Grows the arena to at least `bytes` beyond its kept prefix (the first
// arena_keep bytes, copied into a grown arena).  OPATTR_FAULT=alloc in the
// environment makes growth fail, to exercise the out-of-memory path without
// a GPU fault.
opattr_status ensure_arena(Ctx &c, size_t bytes) {
    bytes += c.arena_keep;
    if (bytes <= c.arena_cap) return OPATTR_OK;
    if (c.arena_fixed) return OPATTR_E_OOM;
    const char *fault = getenv("OPATTR_FAULT");
    if (fault && strcmp(fault, "alloc") == 0) return OPATTR_E_OOM;
    size_t cap = std::max(bytes, (size_t)1 << 20);
    cap = (cap + ((size_t)1 << 20) - 1) & ~(((size_t)1 << 20) - 1);
    if (c.arena && c.arena_keep == 0) {
        // nothing to keep: free first, so the old and new arenas are never held together
        if (cudaStreamSynchronize(c.stream) != cudaSuccess) return cuda_status(c, cudaGetLastError());
        cudaFree(c.arena);
        c.arena = nullptr;
        c.arena_cap = 0;
    }
    char *fresh = nullptr;
    cudaError_t e = cudaMalloc(&fresh, cap);
    if (e == cudaErrorMemoryAllocation) {
        cudaGetLastError();          // clear the sticky-free error state
        return OPATTR_E_OOM;
    }
    if (e != cudaSuccess) return cuda_status(c, e);
    if (c.arena) {
        // the kept prefix moves with the arena
        e = cudaMemcpyAsync(fresh, c.arena, c.arena_keep, cudaMemcpyDeviceToDevice, c.stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(c.stream);
        if (e != cudaSuccess) {
            cudaFree(fresh);
            return cuda_status(c, e);
        }
        if (c.join_korder) c.join_korder = reinterpret_cast<uint32_t *>(fresh + (reinterpret_cast<char *>(c.join_korder) - c.arena));
        cudaFree(c.arena);
    }
    c.arena = fresh;
    c.arena_cap = cap;
    return OPATTR_OK;
}

opattr_status ensure_side(Ctx &c) {
    if (c.side) return OPATTR_OK;
    cudaStream_t s = nullptr;
    cudaEvent_t e[3] = {nullptr, nullptr, nullptr};
    bool ok = cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) == cudaSuccess;
    for (int i = 0; i < 3 && ok; ++i) ok = cudaEventCreateWithFlags(&e[i], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
        cudaGetLastError();
        for (cudaEvent_t x : e)
            if (x) cudaEventDestroy(x);
        if (s) cudaStreamDestroy(s);
        return OPATTR_E_CUDA;
    }
    c.side = s;
    c.ev_fork = e[0];
    c.ev_join = e[1];
    c.ev_join2 = e[2];
    return OPATTR_OK;
}

// Up to SMALL_COPIES transfers in one launch, each between mapped pinned host
// memory and device memory: words when both ends and the size are 4-byte
// aligned (every caller's case), bytes otherwise.
constexpr int SMALL_COPIES = 4;
struct SmallCopies {
    const unsigned char *src[SMALL_COPIES];
    unsigned char *dst[SMALL_COPIES];
    unsigned long long n[SMALL_COPIES];
    int count;
};
__global__ void k_copy_small(SmallCopies cp) {
    pdl_wait();
    const size_t t0 = (size_t)blockIdx.x * blockDim.x + threadIdx.x, step = (size_t)gridDim.x * blockDim.x;
    for (int q = 0; q < cp.count; ++q) {
        const unsigned char *src = cp.src[q];
        unsigned char *dst = cp.dst[q];
        const size_t n = cp.n[q];
        if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst) | n) & 3u) == 0) {
            const uint32_t *s = reinterpret_cast<const uint32_t *>(src);
            uint32_t *d = reinterpret_cast<uint32_t *>(dst);
            for (size_t i = t0; i < n / 4; i += step) d[i] = s[i];
        } else {
            for (size_t i = t0; i < n; i += step) dst[i] = src[i];
        }
    }
}

opattr_status copy_small_n(Ctx &c, int count, const SmallCopy *cp, cudaMemcpyKind kind) {
    if (count <= 0) return OPATTR_OK;
    if (!c.host_mapped) {
        for (int q = 0; q < count; ++q) {
            if (cp[q].bytes == 0) continue;
            const cudaError_t e = cudaMemcpyAsync(cp[q].dst, cp[q].src, cp[q].bytes, kind, c.stream);
            if (e != cudaSuccess) return cuda_status(c, e);
        }
        return OPATTR_OK;
    }
    for (int q0 = 0; q0 < count; q0 += SMALL_COPIES) {
        SmallCopies a{};
        size_t most = 0;
        for (int q = q0; q < count && q < q0 + SMALL_COPIES; ++q) {
            a.src[a.count] = static_cast<const unsigned char *>(cp[q].src);
            a.dst[a.count] = static_cast<unsigned char *>(cp[q].dst);
            a.n[a.count] = cp[q].bytes;
            most = std::max(most, cp[q].bytes);
            a.count++;
        }
        launch(c, "small_copy", k_copy_small, dim3(grid_for((int64_t)std::max<size_t>(most, 1), 256 * 16, 8)),
               dim3(256), 0, a);
    }
    return c.last_error == cudaSuccess ? OPATTR_OK : cuda_status(c, c.last_error);
}

opattr_status copy_small(Ctx &c, void *dst, const void *src, size_t bytes, cudaMemcpyKind kind) {
    if (bytes == 0) return OPATTR_OK;
    const SmallCopy cp{dst, src, bytes};
    return copy_small_n(c, 1, &cp, kind);
}

opattr_status reset_status(Ctx &c) {
    return copy_small(c, c.d_status, c.h_init, sizeof(DevStatus), cudaMemcpyHostToDevice);
}

opattr_status read_status(Ctx &c, int n_extra, const SmallCopy *extra) {
    if (c.last_error != cudaSuccess) return cuda_status(c, c.last_error);
    if (n_extra < 0 || n_extra > SMALL_COPIES - 1) return OPATTR_E_INVALID_ARG;
    SmallCopy cp[SMALL_COPIES];
    int n = 0;
    cp[n++] = SmallCopy{c.h_status, c.d_status, sizeof(DevStatus)};
    for (int q = 0; q < n_extra; ++q) cp[n++] = extra[q];
    opattr_status st = copy_small_n(c, n, cp, cudaMemcpyDeviceToHost);
    if (st) return st;
    cudaError_t e = cudaStreamSynchronize(c.stream);
    if (e != cudaSuccess) return cuda_status(c, e);
    if (c.timing) timing_collect(c);
    // a chained prefix that gave up waiting leaves results that do not count
    if (c.h_status->err & ERR_TIMEOUT) return OPATTR_E_TIMEOUT;
    return OPATTR_OK;
}

int timing_slot(Ctx &c, const char *name) {
    for (size_t i = 0; i < c.slots.size(); ++i)
        if (c.slots[i].name == name || strcmp(c.slots[i].name, name) == 0) return (int)i;
    c.slots.push_back(TimingSlot{name, 0.0, 0});
    return (int)c.slots.size() - 1;
}

static cudaEvent_t take_event(Ctx &c) {
    if (!c.event_pool.empty()) {
        cudaEvent_t e = c.event_pool.back();
        c.event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

void timing_begin(Ctx &c, int, cudaEvent_t *e0, cudaEvent_t *e1) {
    *e0 = take_event(c);
    *e1 = take_event(c);
    cudaEventRecord(*e0, c.stream);
}

void timing_end(Ctx &c, int slot, cudaEvent_t e0, cudaEvent_t e1) {
    cudaEventRecord(e1, c.stream);
    c.pending.push_back({slot, {e0, e1}});
}

void timing_collect(Ctx &c) {
    for (auto &p : c.pending) {
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, p.second.first, p.second.second) == cudaSuccess) {
            c.slots[p.first].total_ms += ms;
            c.slots[p.first].launches += 1;
        }
        c.event_pool.push_back(p.second.first);
        c.event_pool.push_back(p.second.second);
    }
    c.pending.clear();
}

// Each call runs with the context's device current and restores the caller's.
struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

}  // namespace opattr

using namespace opattr;

struct opattr_ctx {
    Ctx c;
};

extern "C" {

opattr_status opattr_create(opattr_ctx **out, int device, void *cuda_stream, const opattr_config *cfg) {
    if (!out) return OPATTR_E_INVALID_ARG;
    *out = nullptr;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess) {
        cudaGetLastError();
        return OPATTR_E_CUDA;
    }
    if (device < 0 || device >= ndev) return OPATTR_E_INVALID_ARG;
    opattr_config conf{};
    conf.mismatch = OPATTR_MISMATCH_SKIP_NAME;
    conf.dedup = 1;
    if (cfg) conf = *cfg;
    if ((int)conf.mismatch < 0 || (int)conf.mismatch > 2 || conf.spin_limit < 0) return OPATTR_E_INVALID_ARG;
    DeviceGuard g(device);
    if (!g.ok) return OPATTR_E_CUDA;
    opattr_ctx *x = new (std::nothrow) opattr_ctx();
    if (!x) return OPATTR_E_OOM;
    Ctx &c = x->c;
    c.device = device;
    c.stream = (cudaStream_t)cuda_stream;
    c.cfg = conf;
    bool fail = cudaMalloc(&c.d_status, sizeof(DevStatus)) != cudaSuccess;
    fail = fail || cudaMallocHost(&c.h_status, sizeof(DevStatus)) != cudaSuccess;
    fail = fail || cudaMallocHost(&c.h_init, sizeof(DevStatus)) != cudaSuccess;
    fail = fail || cudaMallocHost(&c.h_levels, sizeof(uint32_t) * (N_LEVELS + 1 + 256)) != cudaSuccess;
    fail = fail || cudaMallocHost(&c.h_stage, STAGE_BYTES) != cudaSuccess;
    if (fail) {
        cudaGetLastError();
        if (c.d_status) cudaFree(c.d_status);
        if (c.h_status) cudaFreeHost(c.h_status);
        if (c.h_init) cudaFreeHost(c.h_init);
        if (c.h_levels) cudaFreeHost(c.h_levels);
        if (c.h_stage) cudaFreeHost(c.h_stage);
        delete x;
        return OPATTR_E_OOM;
    }
    // the pinned buffers are moved by small kernels when the device sees them
    // at their host addresses (unified addressing), by cudaMemcpyAsync if not
    bool mapped = true;
    for (void *h : {(void *)c.h_status, (void *)c.h_init, (void *)c.h_levels, (void *)c.h_stage}) {
        void *dp = nullptr;
        mapped = mapped && cudaHostGetDevicePointer(&dp, h, 0) == cudaSuccess && dp == h;
    }
    cudaGetLastError();
    c.host_mapped = mapped;
    memset(c.h_init, 0, sizeof(DevStatus));
    c.h_init->mm[MM_KSTART_MIN] = LLONG_MAX;
    c.h_init->mm[MM_KSTART_MAX] = LLONG_MIN;
    c.h_init->mm[MM_RSTART_MIN] = LLONG_MAX;
    c.h_init->mm[MM_REND_MAX] = LLONG_MIN;
    *c.h_status = *c.h_init;
    *out = x;
    return OPATTR_OK;
}

// The enclosure's error bits as a status (the order of do_enclose's checks).
static opattr_status status_from_enclose_err(unsigned err) {
    if (err & ERR_DEPTH) return OPATTR_E_DEPTH;
    if (err & ERR_NOT_NESTED) return OPATTR_E_NOT_NESTED;
    return OPATTR_OK;
}

static opattr_status finish(Ctx &c, opattr_status st) {
    if (c.last_error != cudaSuccess) return cuda_status(c, c.last_error);
    if (st == OPATTR_E_CUDA) c.broken = true;
    return st;
}

opattr_status opattr_enclose(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                             int32_t *range_of_kernel, uint8_t *n_op_enclosing) {
    NvtxCall nvtx("opattr_enclose");
    if (!ctx || !kernels || !ranges) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    return finish(c, do_enclose(c, kernels, ranges, range_of_kernel, n_op_enclosing));
}

opattr_status opattr_match(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ncu *ncu,
                           const opattr_dedup *dedup, int32_t *ncu_idx_of_kernel, uint8_t *match_kind,
                           opattr_match_summary *host_summary) {
    NvtxCall nvtx("opattr_match");
    if (!ctx || !kernels || !ncu) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    return finish(c, do_match(c, kernels, ncu, dedup, ncu_idx_of_kernel, match_kind, host_summary));
}

opattr_status opattr_aggregate(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                               const int32_t *range_of_kernel, const opattr_ncu *ncu,
                               const int32_t *ncu_idx_of_kernel, uint32_t n_ops,
                               const opattr_op_aggregates *dev_out, opattr_totals *host_totals) {
    NvtxCall nvtx("opattr_aggregate");
    if (!ctx || !kernels || !ranges || !ncu) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    return finish(c, do_aggregate(c, kernels, ranges, range_of_kernel, ncu, ncu_idx_of_kernel, n_ops, dev_out,
                                  host_totals));
}

opattr_status opattr_join(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                          const opattr_ncu *ncu, const opattr_dedup *dedup, uint32_t n_ops,
                          int32_t *range_of_kernel, uint8_t *n_op_enclosing, int32_t *ncu_idx_of_kernel,
                          uint8_t *match_kind, const opattr_op_aggregates *dev_out,
                          opattr_match_summary *host_summary, opattr_totals *host_totals) {
    NvtxCall nvtx("opattr_join");
    if (!ctx || !kernels || !ranges || !ncu) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    // the enclosure's kernel time order is kept for the matching (arena_keep);
    // every way out of the join drops it
    struct JoinScope {
        Ctx &c;
        explicit JoinScope(Ctx &ctx) : c(ctx) { c.in_join = true; }
        ~JoinScope() {
            if (c.enclose_pending) cudaStreamSynchronize(c.stream);     // an early return: nothing left running
            c.in_join = false;
            c.order_from_enclose = false;
            c.join_korder = nullptr;
            c.arena_keep = 0;
            c.spec_k = 0;
            c.spec_ran = false;
            c.defer_status = false;
            c.enclose_pending = false;
        }
    } scope(c);
    // the matching's identity pairing may run beside the enclosure: rows one
    // for one with the kernels, no layer deduplication, no per-stream rows;
    // then the enclosure's last status read can wait for the aggregation's
    const bool spec = !dedup && !ncu->stream && kernels->n > 0 && kernels->n == ncu->n && kernels->name_id &&
                      ncu->name_id && ncu_idx_of_kernel;
    for (int pass = 0; pass < 2; ++pass) {
        c.enclose_k_sorted = -1;
        c.spec_k = 0;
        c.spec_ran = false;
        c.enclose_pending = false;
        if (spec) {
            c.spec_kname = kernels->name_id;
            c.spec_nname = ncu->name_id;
            c.spec_idx = ncu_idx_of_kernel;
            c.spec_kind = match_kind;
            c.spec_k = kernels->n;
        }
        c.defer_status = spec && pass == 0;
        opattr_status st = finish(c, do_enclose(c, kernels, ranges, range_of_kernel, n_op_enclosing));
        c.defer_status = false;
        if (st < 0) return st;
        c.order_from_enclose = true;
        opattr_status sm =
            finish(c, do_match(c, kernels, ncu, dedup, ncu_idx_of_kernel, match_kind, host_summary));
        c.order_from_enclose = false;
        c.join_korder = nullptr;             // the aggregation needs no time order
        c.arena_keep = 0;
        if (sm < 0) return sm;
        st = finish(c, do_aggregate(c, kernels, ranges, range_of_kernel, ncu, ncu_idx_of_kernel, n_ops, dev_out,
                                    host_totals));
        if (c.enclose_pending) {
            // the enclosure's verdict and the identity pairing's, read with the
            // aggregation's status (read once more if the aggregation stopped
            // before reading it)
            c.enclose_pending = false;
            if (st < 0) {
                const opattr_status s2 = read_status(c);
                if (s2 < 0) return s2;
            }
            if (c.h_status->flags & F_LEVEL_FIXUP) continue;          // redone without deferring
            if (c.h_status->err & (ERR_NOT_NESTED | ERR_DEPTH)) return status_from_enclose_err(c.h_status->err);
            if (st >= 0 && (c.h_status->flags & F_NAMES_DIFFER)) {
                // the names disagree: the matching and the aggregation proper
                c.order_from_enclose = true;
                c.spec_ran = false;
                sm = finish(c, do_match(c, kernels, ncu, dedup, ncu_idx_of_kernel, match_kind, host_summary));
                c.order_from_enclose = false;
                if (sm < 0) return sm;
                st = finish(c, do_aggregate(c, kernels, ranges, range_of_kernel, ncu, ncu_idx_of_kernel, n_ops,
                                            dev_out, host_totals));
            }
        }
        if (st < 0) return st;
        return sm;
    }
    return OPATTR_E_CUDA;
}

opattr_status opattr_attribute(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                               const int32_t *range_of_kernel, const uint8_t *n_op_enclosing, const opattr_corr *corr,
                               const opattr_fusion *fusion, uint32_t n_ops, uint32_t *op_of_kernel, uint8_t *tier,
                               uint32_t *fused_with, uint8_t *is_fused, opattr_attr_summary *host_summary) {
    NvtxCall nvtx("opattr_attribute");
    if (!ctx || !kernels || !ranges) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    return finish(c, do_attribute(c, kernels, ranges, range_of_kernel, n_op_enclosing, corr, fusion, n_ops,
                                  op_of_kernel, tier, fused_with, is_fused, host_summary));
}

opattr_status opattr_rollup(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                            const int32_t *range_of_kernel, const opattr_ncu *ncu, const int32_t *ncu_idx_of_kernel,
                            uint32_t n_ops, const uint32_t *class_of_op, uint32_t n_classes,
                            const opattr_op_aggregates *dev_out) {
    NvtxCall nvtx("opattr_rollup");
    if (!ctx || !kernels || !ranges || !ncu) return OPATTR_E_INVALID_ARG;
    Ctx &c = ctx->c;
    if (c.broken) return OPATTR_E_STATE;
    DeviceGuard g(c.device);
    if (!g.ok) return OPATTR_E_CUDA;
    return finish(c, do_rollup(c, kernels, ranges, range_of_kernel, ncu, ncu_idx_of_kernel, n_ops, class_of_op,
                               n_classes, dev_out));
}

void opattr_destroy(opattr_ctx *ctx) {
    if (!ctx) return;
    Ctx &c = ctx->c;
    {
        DeviceGuard g(c.device);
        cudaStreamSynchronize(c.stream);
        if (c.arena) cudaFree(c.arena);
        if (c.d_status) cudaFree(c.d_status);
        if (c.h_status) cudaFreeHost(c.h_status);
        if (c.h_init) cudaFreeHost(c.h_init);
        if (c.h_levels) cudaFreeHost(c.h_levels);
        if (c.h_stage) cudaFreeHost(c.h_stage);
        for (auto &p : c.pending) {
            cudaEventDestroy(p.second.first);
            cudaEventDestroy(p.second.second);
        }
        for (cudaEvent_t e : c.event_pool) cudaEventDestroy(e);
        if (c.side) {
            cudaStreamSynchronize(c.side);
            cudaEventDestroy(c.ev_fork);
            cudaEventDestroy(c.ev_join);
            cudaEventDestroy(c.ev_join2);
            cudaStreamDestroy(c.side);
        }
        cudaGetLastError();
    }
    delete ctx;
}

const char *opattr_status_string(opattr_status s) {
    switch (s) {
    case OPATTR_OK: return "ok";
    case OPATTR_W_COUNT_MISMATCH: return "warning: kernel-name count mismatch";
    case OPATTR_W_DEDUP_MISMATCH: return "warning: duplicate-layer kernel without representative row";
    case OPATTR_E_INVALID_ARG: return "invalid argument";
    case OPATTR_E_NOT_NESTED: return "ranges are not nested per stream";
    case OPATTR_E_DEPTH: return "range depth above 31";
    case OPATTR_E_COUNT_MISMATCH: return "kernel-name count mismatch";
    case OPATTR_E_CUDA: return "CUDA error";
    case OPATTR_E_OOM: return "out of device memory";
    case OPATTR_E_TIMEOUT: return "device-side wait timed out";
    case OPATTR_E_STATE: return "context unusable after a CUDA error";
    }
    return "unknown status";
}

opattr_status opattr_set_timing(opattr_ctx *ctx, int enable) {
    if (!ctx) return OPATTR_E_INVALID_ARG;
    ctx->c.timing = enable != 0;
    return OPATTR_OK;
}

opattr_status opattr_set_timing_only(opattr_ctx *ctx, const char *kernel) {
    if (!ctx) return OPATTR_E_INVALID_ARG;
    ctx->c.timing_only = kernel ? kernel : "";
    return OPATTR_OK;
}

int opattr_timing_report(opattr_ctx *ctx, const char **names, double *total_ms, int64_t *launches, int cap) {
    if (!ctx) return 0;
    Ctx &c = ctx->c;
    int n = (int)c.slots.size();
    for (int i = 0; i < n && i < cap; ++i) {
        if (names) names[i] = c.slots[i].name;
        if (total_ms) total_ms[i] = c.slots[i].total_ms;
        if (launches) launches[i] = c.slots[i].launches;
    }
    return n;
}

void opattr_timing_reset(opattr_ctx *ctx) {
    if (!ctx) return;
    for (auto &s : ctx->c.slots) { s.total_ms = 0.0; s.launches = 0; }
    ctx->c.launches = 0;
}

int64_t opattr_launch_count(const opattr_ctx *ctx) { return ctx ? ctx->c.launches : 0; }

}  // extern "C"
