// noalloc.cu -- opattr_match without any device allocation.
//
// Some callers must not allocate device memory at all: an attribution pass
// that runs inside the application being profiled (an injection library or a
// profiler callback) has to leave that application's device-memory footprint
// and addresses exactly as they were, and a host whose device memory is owned
// by a caching allocator, or a loop that forbids allocation on its hot path,
// cannot hand out cudaMalloc calls either.  opattr_match_noalloc gives them
// the matching step of the join with all of its scratch -- the status block
// and the sort buffers -- in one file-scope device array of fixed size.  The
// match path itself is the one opattr_match runs.
#include <mutex>

#include "common.cuh"

namespace opattr {
opattr_status do_match(Ctx &c, const opattr_kernels *kern, const opattr_ncu *ncu, const opattr_dedup *dd,
                       int32_t *out_idx, uint8_t *out_kind, opattr_match_summary *sum);
}
using namespace opattr;

// Large enough for OPATTR_MATCH_NOALLOC_MAX kernels and rows on the general
// (sorting) path: 4.8 MB of sort buffers and tables, checked against this size
// on every call (a request beyond it returns OPATTR_E_OOM, never a stray
// access).  Every GPU that loads the library holds it until the process exits.
static constexpr size_t NOALLOC_SCRATCH_BYTES = (size_t)6 << 20;
static __device__ __align__(256) unsigned char g_match_scratch[NOALLOC_SCRATCH_BYTES];

namespace {
std::mutex g_lock;                       // one call at a time: every call shares the array

// Waits for the call's queued work before the lock is released, whatever the
// call returns, so the next caller never reuses the array under it.
struct DrainOnExit {
    cudaStream_t s;
    ~DrainOnExit() {
        cudaStreamSynchronize(s);
        cudaGetLastError();
    }
};
}  // namespace

extern "C" opattr_status opattr_match_noalloc(const opattr_kernels *kernels, const opattr_ncu *ncu,
                                              opattr_mismatch_mode mismatch, int32_t *ncu_idx_of_kernel,
                                              uint8_t *match_kind, opattr_match_summary *host_summary,
                                              void *cuda_stream) {
    if (!kernels || !ncu) return OPATTR_E_INVALID_ARG;
    if ((int)mismatch < 0 || (int)mismatch > 2) return OPATTR_E_INVALID_ARG;
    if (ncu->stream) return OPATTR_E_INVALID_ARG;
    if (kernels->n < 0 || ncu->n < 0 || kernels->n > OPATTR_MATCH_NOALLOC_MAX || ncu->n > OPATTR_MATCH_NOALLOC_MAX)
        return OPATTR_E_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return OPATTR_E_CUDA;
    }
    std::lock_guard<std::mutex> guard(g_lock);
    // The array's device address in the CUDA context current now (the
    // host-side name is only a stand-in for it).  Looked up on every call: an
    // address kept from an earlier call would belong to a context that a
    // device reset has destroyed, or to another context of the same device.
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_match_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return OPATTR_E_CUDA;
    }
    char *base = static_cast<char *>(p);
    // status block first, the arena after it; host mirrors are plain host memory
    DevStatus h_status, h_init;
    memset(&h_init, 0, sizeof h_init);
    h_init.mm[MM_KSTART_MIN] = LLONG_MAX;
    h_init.mm[MM_KSTART_MAX] = LLONG_MIN;
    h_init.mm[MM_RSTART_MIN] = LLONG_MAX;
    h_init.mm[MM_REND_MAX] = LLONG_MIN;
    h_status = h_init;
    Ctx c;
    c.device = dev;
    c.stream = (cudaStream_t)cuda_stream;
    c.cfg.mismatch = mismatch;
    c.cfg.dedup = 0;
    c.d_status = reinterpret_cast<DevStatus *>(base);
    c.h_status = &h_status;
    c.h_init = &h_init;
    const size_t status_bytes = (sizeof(DevStatus) + 255) & ~(size_t)255;
    c.arena = base + status_bytes;
    c.arena_cap = NOALLOC_SCRATCH_BYTES - status_bytes;
    c.arena_fixed = true;
    DrainOnExit drain{c.stream};
    opattr_status st = do_match(c, kernels, ncu, nullptr, ncu_idx_of_kernel, match_kind, host_summary);
    if (c.last_error != cudaSuccess) return OPATTR_E_CUDA;
    return st;
}
