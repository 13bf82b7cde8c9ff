// util.cu -- kernel time-order check and permutation.
#include "sort.cuh"
#include "util.cuh"

namespace opattr {

constexpr int CHK_THREADS = 256;

// Tiles of CHK_TILE consecutive kernels (the digit passes' tiles), a block
// at a time, each thread taking two groups of eight consecutive kernels per
// tile (16-byte loads when the arrays allow) and comparing each (start,
// stream) with its successor; min / max and the order flag are reduced per
// block and published with one atomic each.  With stream_hist the block also
// counts the kernels of each stream (added to the 256 counters once per
// block), and with tile_hist it writes each tile's counts as column `tile`
// of a stream-major matrix (tile_hist[s * ntiles + tile]): the digit
// histogram of a stable partition by stream, in array order.
constexpr int CHK_G = 8;
constexpr int CHK_TILE = 2 * CHK_THREADS * CHK_G;
static_assert(CHK_TILE == RADIX_TILE, "the order check's tiles are the digit passes' tiles");
__global__ void __launch_bounds__(CHK_THREADS) k_check_kernel_order(const uint8_t *__restrict__ stream,
                                                                    const int64_t *__restrict__ start, int64_t n,
                                                                    int vec, DevStatus *st,
                                                                    uint32_t *__restrict__ stream_hist,
                                                                    uint32_t *__restrict__ tile_hist) {
    pdl_wait();
    __shared__ long long smin[CHK_THREADS / 32], smax[CHK_THREADS / 32];
    __shared__ int sbad[CHK_THREADS / 32];
    __shared__ uint32_t sh[256], th[256];
    const bool count = stream_hist || tile_hist;
    for (int i = threadIdx.x; i < 256; i += CHK_THREADS) sh[i] = th[i] = 0;
    __syncthreads();
    long long mn = LLONG_MAX, mx = LLONG_MIN;
    int unsorted = 0;
    const int64_t ntiles = (n + CHK_TILE - 1) / CHK_TILE;
    for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        for (int r = 0; r < 2; ++r) {
            const int64_t i0 = (tile * (CHK_TILE / CHK_G) + r * CHK_THREADS + threadIdx.x) * CHK_G;
            if (i0 >= n) continue;
            long long t[CHK_G + 1];
            unsigned s[CHK_G + 1];
            if (vec && i0 + CHK_G <= n) {
                const longlong2 *p = reinterpret_cast<const longlong2 *>(start + i0);
#pragma unroll
                for (int q = 0; q < CHK_G / 2; ++q) {
                    const longlong2 x = p[q];
                    t[2 * q] = x.x;
                    t[2 * q + 1] = x.y;
                }
                const uint2 w = *reinterpret_cast<const uint2 *>(stream + i0);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    s[u] = (w.x >> (8 * u)) & 0xFFu;
                    s[4 + u] = (w.y >> (8 * u)) & 0xFFu;
                }
            } else {
#pragma unroll
                for (int u = 0; u < CHK_G; ++u) {
                    t[u] = i0 + u < n ? start[i0 + u] : LLONG_MAX;
                    s[u] = i0 + u < n ? stream[i0 + u] : 255u;
                }
            }
            t[CHK_G] = i0 + CHK_G < n ? start[i0 + CHK_G] : LLONG_MAX;
            s[CHK_G] = i0 + CHK_G < n ? stream[i0 + CHK_G] : 255u;
#pragma unroll
            for (int u = 0; u < CHK_G; ++u) {
                if (i0 + u >= n) break;
                mn = t[u] < mn ? t[u] : mn;
                mx = t[u] > mx ? t[u] : mx;
                if (i0 + u + 1 < n) unsorted |= (t[u + 1] < t[u]) || (t[u + 1] == t[u] && s[u + 1] < s[u]);
                if (count) atomicAdd(&th[s[u]], 1u);
            }
        }
        if (count) {
            __syncthreads();
            for (int i = threadIdx.x; i < 256; i += CHK_THREADS) {
                const uint32_t x = th[i];
                if (tile_hist) tile_hist[(int64_t)i * ntiles + tile] = x;
                sh[i] += x;
                th[i] = 0;
            }
            __syncthreads();
        }
    }
    if (stream_hist) {
        for (int i = threadIdx.x; i < 256; i += CHK_THREADS)
            if (sh[i]) atomicAdd(&stream_hist[i], sh[i]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        long long a = __shfl_xor_sync(0xffffffffu, mn, o), b = __shfl_xor_sync(0xffffffffu, mx, o);
        mn = a < mn ? a : mn;
        mx = b > mx ? b : mx;
    }
    unsorted = __any_sync(0xffffffffu, unsorted);
    if (lane_id() == 0) {
        smin[threadIdx.x >> 5] = mn;
        smax[threadIdx.x >> 5] = mx;
        sbad[threadIdx.x >> 5] = unsorted;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int bad = 0;
        for (int w = 0; w < CHK_THREADS / 32; ++w) {
            mn = smin[w] < mn ? smin[w] : mn;
            mx = smax[w] > mx ? smax[w] : mx;
            bad |= sbad[w];
        }
        atomicMin(&st->mm[MM_KSTART_MIN], mn);
        atomicMax(&st->mm[MM_KSTART_MAX], mx);
        if (bad) set_flag(st, F_K_UNSORTED);
    }
}

void check_kernel_order(Ctx &c, const uint8_t *stream, const int64_t *start, int64_t n, uint32_t *stream_hist,
                        uint32_t *tile_hist) {
    if (n <= 0) return;
    const int vec = ((reinterpret_cast<uintptr_t>(start) & 15) == 0) && ((reinterpret_cast<uintptr_t>(stream) & 7) == 0);
    launch(c, "check_kernel_order", k_check_kernel_order, dim3(grid_for(n, CHK_TILE, REDUCE_GRID)),
           dim3(CHK_THREADS), 0, stream, start, n, vec, c.d_status, stream_hist, tile_hist);
}

__global__ void k_time_keys(const uint8_t *__restrict__ stream, const int64_t *__restrict__ start, int64_t n,
                            long long tmin, const uint8_t *__restrict__ scmap, int sbits,
                            uint64_t *__restrict__ keys) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const unsigned s = scmap ? scmap[stream[i]] : stream[i];
        keys[i] = ((uint64_t)(start[i] - tmin) << sbits) | s;
    }
}

size_t kernel_order_scratch(int64_t n) {
    Need nd;
    nd.add<uint64_t>(n).add<uint64_t>(n).add<uint32_t>(n).add<uint32_t>(n);
    nd.add<uint32_t>(radix_hist_elems(n)).add<uint32_t>(scan_scratch_elems(radix_hist_elems(n)));
    return nd.bytes;
}

uint32_t *kernel_time_order(Ctx &c, Arena &a, const uint8_t *stream, const int64_t *start, int64_t n,
                            const uint8_t *scmap, int stream_bits) {
    uint64_t *k0 = a.take<uint64_t>(n), *k1 = a.take<uint64_t>(n);
    uint32_t *v0 = a.take<uint32_t>(n), *v1 = a.take<uint32_t>(n);
    uint32_t *hist = a.take<uint32_t>(radix_hist_elems(n));
    uint32_t *part = a.take<uint32_t>(scan_scratch_elems(radix_hist_elems(n)));
    if (!k0 || !k1 || !v0 || !v1 || !hist || !part) return nullptr;
    long long tmin = c.h_status->mm[MM_KSTART_MIN], tmax = c.h_status->mm[MM_KSTART_MAX];
    const int sbits = scmap ? stream_bits : 8;
    launch(c, "time_keys", k_time_keys, dim3(grid_for(n, 256, 65535)), dim3(256), 0, stream, start, n, tmin, scmap,
           sbits, k0);
    uint64_t *ko;
    uint32_t *vo;
    radix_sort_pairs<uint64_t>(c, k0, v0, k1, v1, n, bits_for((uint64_t)(tmax - tmin)) + sbits, true, hist, part,
                               &ko, &vo);
    return vo;
}

}  // namespace opattr
