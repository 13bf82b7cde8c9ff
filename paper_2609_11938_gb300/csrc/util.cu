// util.cu -- kernel time-order check and permutation.
#include "sort.cuh"
#include "util.cuh"

namespace opattr {

constexpr int CHK_THREADS = 256;
constexpr int CHK_ITEMS = 8;

// Each thread checks CHK_ITEMS consecutive pairs (i, i+1); loads are
// coalesced across the block.
__global__ void __launch_bounds__(CHK_THREADS) k_check_kernel_order(const uint8_t *__restrict__ stream,
                                                                    const int64_t *__restrict__ start, int64_t n,
                                                                    DevStatus *st) {
    __shared__ long long smin[CHK_THREADS / 32], smax[CHK_THREADS / 32];
    __shared__ int bad;
    if (threadIdx.x == 0) bad = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * CHK_THREADS * CHK_ITEMS;
    long long mn = LLONG_MAX, mx = LLONG_MIN;
    int unsorted = 0;
#pragma unroll
    for (int it = 0; it < CHK_ITEMS; ++it) {
        int64_t i = base + it * CHK_THREADS + threadIdx.x;
        if (i < n) {
            long long t = start[i];
            mn = t < mn ? t : mn;
            mx = t > mx ? t : mx;
            if (i + 1 < n) {
                long long u = start[i + 1];
                unsorted |= (u < t) || (u == t && stream[i + 1] < stream[i]);
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        long long a = __shfl_xor_sync(0xffffffffu, mn, o), b = __shfl_xor_sync(0xffffffffu, mx, o);
        mn = a < mn ? a : mn;
        mx = b > mx ? b : mx;
    }
    if (unsorted) bad = 1;
    if (lane_id() == 0) { smin[threadIdx.x >> 5] = mn; smax[threadIdx.x >> 5] = mx; }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < CHK_THREADS / 32; ++w) {
            mn = smin[w] < mn ? smin[w] : mn;
            mx = smax[w] > mx ? smax[w] : mx;
        }
        mn = smin[0] < mn ? smin[0] : mn;
        mx = smax[0] > mx ? smax[0] : mx;
        atomicMin(&st->mm[MM_KSTART_MIN], mn);
        atomicMax(&st->mm[MM_KSTART_MAX], mx);
        if (bad) set_flag(st, F_K_UNSORTED);
    }
}

void check_kernel_order(Ctx &c, const uint8_t *stream, const int64_t *start, int64_t n) {
    if (n <= 0) return;
    launch(c, "check_kernel_order", k_check_kernel_order, dim3(grid_for(n, CHK_THREADS * CHK_ITEMS)),
           dim3(CHK_THREADS), 0, stream, start, n, c.d_status);
}

__global__ void k_time_keys(const uint8_t *__restrict__ stream, const int64_t *__restrict__ start, int64_t n,
                            long long tmin, uint64_t *__restrict__ keys) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        keys[i] = ((uint64_t)(start[i] - tmin) << 8) | stream[i];
}

size_t kernel_order_scratch(int64_t n) {
    Need nd;
    nd.add<uint64_t>(n).add<uint64_t>(n).add<uint32_t>(n).add<uint32_t>(n);
    nd.add<uint32_t>(radix_hist_elems(n)).add<uint32_t>(scan_scratch_elems(radix_hist_elems(n)));
    return nd.bytes;
}

uint32_t *kernel_time_order(Ctx &c, Arena &a, const uint8_t *stream, const int64_t *start, int64_t n) {
    uint64_t *k0 = a.take<uint64_t>(n), *k1 = a.take<uint64_t>(n);
    uint32_t *v0 = a.take<uint32_t>(n), *v1 = a.take<uint32_t>(n);
    uint32_t *hist = a.take<uint32_t>(radix_hist_elems(n));
    uint32_t *part = a.take<uint32_t>(scan_scratch_elems(radix_hist_elems(n)));
    if (!k0 || !k1 || !v0 || !v1 || !hist || !part) return nullptr;
    long long tmin = c.h_status->mm[MM_KSTART_MIN], tmax = c.h_status->mm[MM_KSTART_MAX];
    launch(c, "time_keys", k_time_keys, dim3(grid_for(n, 256, 65535)), dim3(256), 0, stream, start, n, tmin, k0);
    uint64_t *ko;
    uint32_t *vo;
    radix_sort_pairs<uint64_t>(c, k0, v0, k1, v1, n, bits_for((uint64_t)(tmax - tmin)) + 8, true, hist, part, &ko,
                               &vo);
    return vo;
}

}  // namespace opattr
