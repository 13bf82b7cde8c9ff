// sort.cu -- device-wide exclusive scan and a stable LSD radix sort with
// warp-level digit ranking.
//
// A scan out of place is one pass: tiles chain their prefixes by decoupled
// look-back (warp_lookback_exclusive in sort.cuh, a bounded wait on tiles
// that started earlier); a scan in place is three launches with no waits.  A
// radix sort pass is three launches (tile histograms -> single-pass scan of
// the histogram matrix, out of place -> scatter).
#include <cstdlib>
#include <cstring>

#include "sort.cuh"

namespace opattr {

// ------------------------------------------------------------------ scan, in place
// Three launches (tile sums, their scan, the tiles), no block waits on another:
// the scan of a buffer onto itself, where the single pass below could not
// fall back on the input.
// Each warp owns 512 consecutive elements and walks them 32 at a time
// (coalesced), carrying its running sum.
__global__ void __launch_bounds__(SCAN_THREADS) k_scan_reduce(const uint32_t *__restrict__ in, int64_t n,
                                                              uint32_t *__restrict__ partials) {
    pdl_wait();
    __shared__ uint32_t wbuf[33];
    const int64_t base = (int64_t)blockIdx.x * SCAN_TILE + (threadIdx.x >> 5) * (SCAN_TILE / 8);
    uint32_t s = 0;
#pragma unroll
    for (int it = 0; it < SCAN_ITEMS; ++it) {
        int64_t i = base + it * 32 + lane_id();
        if (i < n) s += in[i];
    }
    uint32_t tot = block_sum<uint32_t>(s, wbuf);
    if (threadIdx.x == 0) partials[blockIdx.x] = tot;
}

// One block scans the tile sums (exclusive) in place; partials[nt] = total.
__global__ void __launch_bounds__(1024) k_scan_partials(uint32_t *partials, int64_t nt, uint32_t *total_dev) {
    pdl_wait();
    __shared__ uint32_t wbuf[33];
    uint32_t carry = 0;
    for (int64_t b = 0; b < nt; b += 1024) {
        int64_t i = b + threadIdx.x;
        uint32_t v = i < nt ? partials[i] : 0u;
        uint32_t tot;
        uint32_t ex = block_exclusive_scan<uint32_t>(v, wbuf, &tot);
        if (i < nt) partials[i] = carry + ex;
        carry += tot;
    }
    if (threadIdx.x == 0) {
        partials[nt] = carry;
        if (total_dev) *total_dev = carry;
    }
}

__global__ void __launch_bounds__(SCAN_THREADS) k_scan_down(const uint32_t *in, uint32_t *out, int64_t n,
                                                            const uint32_t *__restrict__ partials) {
    pdl_wait();
    __shared__ uint32_t wbuf[33];
    const unsigned w = threadIdx.x >> 5;
    const int64_t base = (int64_t)blockIdx.x * SCAN_TILE + w * (SCAN_TILE / 8);
    uint32_t v[SCAN_ITEMS];
    uint32_t carry = 0;
#pragma unroll
    for (int it = 0; it < SCAN_ITEMS; ++it) {
        int64_t i = base + it * 32 + lane_id();
        uint32_t x = i < n ? in[i] : 0u;
        uint32_t inc = warp_inclusive_scan(x);
        v[it] = carry + inc - x;
        carry += __shfl_sync(0xffffffffu, inc, 31);
    }
    // carry = this warp's total; block-exclusive prefix over warps
    uint32_t wtot;
    uint32_t wpre = block_exclusive_scan<uint32_t>(lane_id() == 0 ? carry : 0u, wbuf, &wtot);
    wpre = __shfl_sync(0xffffffffu, wpre, 0);
    const uint32_t off = partials[blockIdx.x] + wpre;
#pragma unroll
    for (int it = 0; it < SCAN_ITEMS; ++it) {
        int64_t i = base + it * 32 + lane_id();
        if (i < n) out[i] = off + v[it];
    }
}

// ------------------------------------------------------------------ scan
// One pass: a block takes the next tile of SCAN_TILE elements (tiles in the
// order blocks start), each warp scans 512 consecutive elements 32 at a time
// (coalesced) carrying its running sum, the warp totals are scanned across
// the block, and the tile's offset comes from the chained prefix of the tiles
// before it.  Out of place only: a tile whose wait gives up sums the input of
// the tiles before it that are still silent.
__global__ void __launch_bounds__(SCAN_THREADS) k_scan_onepass(const uint32_t *__restrict__ in,
                                                               uint32_t *__restrict__ out, int64_t n,
                                                               unsigned long long *status, unsigned *tile_ctr,
                                                               int64_t nt, uint32_t *total_dev, int64_t spin_limit,
                                                               int fault, DevStatus *st) {
    pdl_wait();
    __shared__ uint32_t wbuf[33];
    __shared__ unsigned tile_s;
    __shared__ uint32_t off_s;
    if (threadIdx.x == 0) tile_s = atomicAdd(tile_ctr, 1u);
    __syncthreads();
    const int64_t tile = tile_s;
    const unsigned w = threadIdx.x >> 5;
    const int64_t base = tile * SCAN_TILE + w * (SCAN_TILE / 8);
    uint32_t v[SCAN_ITEMS];
    uint32_t carry = 0;
#pragma unroll
    for (int it = 0; it < SCAN_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane_id();
        const uint32_t x = i < n ? in[i] : 0u;
        const uint32_t inc = warp_inclusive_scan(x);
        v[it] = carry + inc - x;
        carry += __shfl_sync(0xffffffffu, inc, 31);
    }
    // carry = this warp's total; block-exclusive prefix over warps
    uint32_t btot;
    uint32_t wpre = block_exclusive_scan<uint32_t>(lane_id() == 0 ? carry : 0u, wbuf, &btot);
    wpre = __shfl_sync(0xffffffffu, wpre, 0);
    if (threadIdx.x < 32) {
        const uint32_t ex = warp_lookback_exclusive(status, tile, btot, in, n, SCAN_TILE, spin_limit, fault != 0, st);
        if (threadIdx.x == 0) {
            off_s = ex;
            if (tile == nt - 1 && total_dev) *total_dev = ex + btot;
        }
    }
    __syncthreads();
    const uint32_t off = off_s + wpre;
#pragma unroll
    for (int it = 0; it < SCAN_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane_id();
        if (i < n) out[i] = off + v[it];
    }
}

// Small scans in one block (one launch instead of three): each of the 32
// warps scans a contiguous run of 1,024 elements in 32 coalesced rounds,
// carrying the running total in registers; one barrier exchanges the warp
// totals.  Every element is read and written by the same thread, so the
// scan may run in place.
constexpr int64_t SCAN_ONE_BLOCK = 32 * 1024;
__global__ void __launch_bounds__(1024) k_scan_small(const uint32_t *in, uint32_t *out, int64_t n,
                                                     uint32_t *total_dev) {
    pdl_wait();
    __shared__ uint32_t wsum[32];
    const unsigned w = threadIdx.x >> 5, lane = lane_id();
    const int64_t b = (int64_t)w * 1024 + lane;
    uint32_t v[32];
#pragma unroll
    for (int r = 0; r < 32; ++r) v[r] = b + r * 32 < n ? in[b + r * 32] : 0u;
    uint32_t carry = 0;
#pragma unroll
    for (int r = 0; r < 32; ++r) {
        const uint32_t inc = warp_inclusive_scan(v[r]);
        const uint32_t ex = carry + inc - v[r];
        carry += __shfl_sync(0xffffffffu, inc, 31);
        v[r] = ex;
    }
    if (lane == 0) wsum[w] = carry;
    __syncthreads();
    const uint32_t x = wsum[lane];
    const uint32_t xs = warp_inclusive_scan(x);
    const uint32_t base = __shfl_sync(0xffffffffu, xs - x, (int)w);
    const uint32_t tot = __shfl_sync(0xffffffffu, xs, 31);
#pragma unroll
    for (int r = 0; r < 32; ++r)
        if (b + r * 32 < n) out[b + r * 32] = base + v[r];
    if (threadIdx.x == 0 && total_dev) *total_dev = tot;
}

void scan_exclusive_u32(Ctx &c, const uint32_t *in, uint32_t *out, int64_t n, uint32_t *partials,
                        uint32_t *total_dev) {
    int64_t nt = (n + SCAN_TILE - 1) / SCAN_TILE;
    if (n <= 0) {
        if (total_dev) cudaMemsetAsync(total_dev, 0, sizeof(uint32_t), c.stream);
        return;
    }
    if (n <= SCAN_ONE_BLOCK) {
        launch(c, "scan_small", k_scan_small, dim3(1), dim3(1024), 0, in, out, n, total_dev);
        return;
    }
    if (in == out) {
        launch(c, "scan_reduce", k_scan_reduce, dim3((unsigned)nt), dim3(SCAN_THREADS), 0, in, n, partials);
        launch(c, "scan_partials", k_scan_partials, dim3(1), dim3(1024), 0, partials, nt, total_dev);
        launch(c, "scan_down", k_scan_down, dim3((unsigned)nt), dim3(SCAN_THREADS), 0, in, out, n,
               (const uint32_t *)partials);
        return;
    }
    unsigned long long *status = reinterpret_cast<unsigned long long *>(partials);
    cudaMemsetAsync(status, 0, sizeof(unsigned long long) * (nt + 1), c.stream);
    const char *fault = getenv("OPATTR_FAULT");
    const int lb_fault = fault && strcmp(fault, "lookback") == 0;
    const int64_t spin = c.cfg.spin_limit > 0 ? c.cfg.spin_limit : LB_SPIN_DEFAULT;
    launch(c, "scan", k_scan_onepass, dim3((unsigned)nt), dim3(SCAN_THREADS), 0, in, out, n, status,
           reinterpret_cast<unsigned *>(status + nt), nt, total_dev, spin, lb_fault, c.d_status);
}

// ------------------------------------------------------------------ radix sort
template <typename K>
__device__ __forceinline__ unsigned digit_of(K key, int shift) {
    return (unsigned)(key >> shift) & (RADIX_BINS - 1);
}

// Per tile, the count of each digit; hist is digit-major: hist[d * ntiles + tile].
template <typename K>
__global__ void __launch_bounds__(RADIX_THREADS) k_radix_upsweep(const K *__restrict__ keys, int64_t n, int shift,
                                                                 uint32_t *__restrict__ hist, int64_t ntiles) {
    pdl_wait();
    __shared__ uint32_t h[RADIX_THREADS / 32][RADIX_BINS];
    const unsigned w = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) (&h[0][0])[i] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RADIX_TILE + w * (RADIX_TILE / 8);
#pragma unroll 4
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        int64_t i = base + it * 32 + lane_id();
        if (i < n) atomicAdd(&h[w][digit_of(keys[i], shift)], 1u);
    }
    __syncthreads();
    for (int d = threadIdx.x; d < RADIX_BINS; d += RADIX_THREADS) {
        uint32_t s = 0;
#pragma unroll
        for (int q = 0; q < RADIX_THREADS / 32; ++q) s += h[q][d];
        hist[(int64_t)d * ntiles + blockIdx.x] = s;
    }
}

// Stable scatter of one tile.  Warp w ranks its 512 keys in order, 32 at a
// time, with peer groups from one ballot per digit bit; per-(warp, digit) counts give the
// tile-local order; keys are staged in shared memory sorted by digit and
// then written out so equal-digit runs go to consecutive addresses.
template <typename K>
__global__ void __launch_bounds__(RADIX_THREADS) k_radix_downsweep(const K *__restrict__ kin,
                                                                   const uint32_t *__restrict__ vin,
                                                                   K *__restrict__ kout, uint32_t *__restrict__ vout,
                                                                   int64_t n, int shift,
                                                                   const uint32_t *__restrict__ offs,
                                                                   int64_t ntiles) {
    pdl_wait();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    K *ks = reinterpret_cast<K *>(smem_raw);
    uint32_t *vs = reinterpret_cast<uint32_t *>(ks + RADIX_TILE);
    uint32_t *wcnt = vs + RADIX_TILE;                          // [8][256]
    uint32_t *dstart = wcnt + (RADIX_THREADS / 32) * RADIX_BINS; // [256] tile-local digit start
    uint32_t *gbase = dstart + RADIX_BINS;                      // [256] global start of digit run
    uint32_t *wbuf = gbase + RADIX_BINS;                        // [33]
    const unsigned w = threadIdx.x >> 5, lane = lane_id();
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) wcnt[i] = 0;
    __syncthreads();

    const int64_t tile0 = (int64_t)blockIdx.x * RADIX_TILE;
    const int64_t base = tile0 + w * (RADIX_TILE / 8);
    K key[RADIX_ITEMS];
    uint32_t val[RADIX_ITEMS];
    uint32_t rank[RADIX_ITEMS];
    const unsigned lt = lanemask_lt();
    unsigned peers[RADIX_ITEMS];
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {        // keys, digits and peer groups first: independent
        int64_t i = base + it * 32 + lane;
        bool ok = i < n;
        key[it] = ok ? kin[i] : K(0);
        val[it] = ok ? (vin ? vin[i] : (uint32_t)i) : 0u;
    }
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const bool ok = base + it * 32 + lane < n;
        const unsigned d = ok ? digit_of(key[it], shift) : RADIX_BINS;    // RADIX_BINS = no key
        peers[it] = warp_peers8(d, ok);
    }
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const bool ok = base + it * 32 + lane < n;
        const unsigned d = ok ? digit_of(key[it], shift) : RADIX_BINS;
        unsigned before = d < RADIX_BINS ? wcnt[w * RADIX_BINS + d] : 0u;
        __syncwarp();
        if (d < RADIX_BINS && (peers[it] & lt) == 0) wcnt[w * RADIX_BINS + d] = before + __popc(peers[it]);
        __syncwarp();
        rank[it] = before + __popc(peers[it] & lt);
    }
    __syncthreads();
    // per digit: exclusive prefix over warps, then over digits
    uint32_t tot = 0;
    for (int d = threadIdx.x; d < RADIX_BINS; d += RADIX_THREADS) {
        uint32_t s = 0;
#pragma unroll
        for (int q = 0; q < RADIX_THREADS / 32; ++q) {
            uint32_t x = wcnt[q * RADIX_BINS + d];
            wcnt[q * RADIX_BINS + d] = s;
            s += x;
        }
        tot = s;
    }
    // RADIX_THREADS == RADIX_BINS: thread d holds digit d's tile count
    uint32_t ds = block_exclusive_scan<uint32_t>(threadIdx.x < RADIX_BINS ? tot : 0u, wbuf, (uint32_t *)nullptr);
    if (threadIdx.x < RADIX_BINS) {
        dstart[threadIdx.x] = ds;
        gbase[threadIdx.x] = offs[(int64_t)threadIdx.x * ntiles + blockIdx.x];
    }
    __syncthreads();
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        int64_t i = base + it * 32 + lane;
        if (i < n) {
            unsigned d = digit_of(key[it], shift);
            uint32_t p = dstart[d] + wcnt[w * RADIX_BINS + d] + rank[it];
            ks[p] = key[it];
            vs[p] = val[it];
        }
    }
    __syncthreads();
    int64_t cnt = n - tile0 < RADIX_TILE ? n - tile0 : RADIX_TILE;
    for (int i = threadIdx.x; i < cnt; i += RADIX_THREADS) {
        K k = ks[i];
        unsigned d = digit_of(k, shift);
        int64_t o = (int64_t)gbase[d] + (i - dstart[d]);
        kout[o] = k;
        vout[o] = vs[i];
    }
}

template <typename K>
static size_t downsweep_smem() {
    return (size_t)RADIX_TILE * (sizeof(K) + 4) + ((RADIX_THREADS / 32) * RADIX_BINS + 2 * RADIX_BINS + 33) * 4;
}

template <typename K>
void radix_sort_pairs(Ctx &c, K *k0, uint32_t *v0, K *k1, uint32_t *v1, int64_t n, int bits, bool iota,
                      uint32_t *hist, uint32_t *partials, K **kout, uint32_t **vout) {
    static unsigned attr_done = 0;   // one bit per device
    if (c.device < 32 && !(attr_done & (1u << c.device))) {
        cudaFuncSetAttribute(k_radix_downsweep<K>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)downsweep_smem<K>());
        attr_done |= 1u << c.device;
    }
    K *ka = k0, *kb = k1;
    uint32_t *va = v0, *vb = v1;
    const int64_t ntiles = (n + RADIX_TILE - 1) / RADIX_TILE;
    // the tiles' digit counts, then their scan (out of place, one pass)
    uint32_t *hcount = hist, *hoff = hist + ntiles * RADIX_BINS;
    if (iota && bits <= 0) bits = 1;   // equal keys: one pass still writes the indices
    for (int shift = 0; shift < bits && n > 0; shift += RADIX_BITS) {
        const bool first = shift == 0;
        launch(c, "radix_upsweep", k_radix_upsweep<K>, dim3((unsigned)ntiles), dim3(RADIX_THREADS), 0,
               (const K *)ka, n, shift, hcount, ntiles);
        scan_exclusive_u32(c, hcount, hoff, ntiles * RADIX_BINS, partials, nullptr);
        launch(c, "radix_downsweep", k_radix_downsweep<K>, dim3((unsigned)ntiles), dim3(RADIX_THREADS),
               downsweep_smem<K>(), (const K *)ka, (const uint32_t *)((first && iota) ? nullptr : va), kb, vb, n,
               shift, (const uint32_t *)hoff, ntiles);
        K *tk = ka; ka = kb; kb = tk;
        uint32_t *tv = va; va = vb; vb = tv;
    }
    *kout = ka;
    *vout = va;
}

template void radix_sort_pairs<uint32_t>(Ctx &, uint32_t *, uint32_t *, uint32_t *, uint32_t *, int64_t, int, bool,
                                         uint32_t *, uint32_t *, uint32_t **, uint32_t **);
template void radix_sort_pairs<uint8_t>(Ctx &, uint8_t *, uint32_t *, uint8_t *, uint32_t *, int64_t, int, bool,
                                        uint32_t *, uint32_t *, uint8_t **, uint32_t **);
template void radix_sort_pairs<uint64_t>(Ctx &, uint64_t *, uint32_t *, uint64_t *, uint32_t *, int64_t, int, bool,
                                         uint32_t *, uint32_t *, uint64_t **, uint32_t **);

}  // namespace opattr
