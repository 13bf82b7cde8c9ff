// sort.cuh -- device-wide exclusive scan and stable LSD radix sort (host side).
#pragma once
#include "common.cuh"

namespace opattr {

constexpr int SCAN_THREADS = 256;
constexpr int SCAN_ITEMS = 16;
constexpr int SCAN_TILE = SCAN_THREADS * SCAN_ITEMS;     // 4096 elements per block

constexpr int RADIX_THREADS = 256;
constexpr int RADIX_ITEMS = 16;
constexpr int RADIX_TILE = RADIX_THREADS * RADIX_ITEMS;  // 4096 keys per block
constexpr int RADIX_BITS = 8;
constexpr int RADIX_BINS = 1 << RADIX_BITS;

// Scratch for a scan of n elements (u32 units): one 64-bit status word per
// tile of the single-pass scan and the tile counter.
inline int64_t scan_scratch_elems(int64_t n) { return 2 * ((n + SCAN_TILE - 1) / SCAN_TILE) + 4; }

// out[i] = in[0] + ... + in[i-1]; *total_dev (device, may be NULL) = sum of all.
// in and out may alias.  `partials` holds scan_scratch_elems(n) u32.
void scan_exclusive_u32(Ctx &c, const uint32_t *in, uint32_t *out, int64_t n, uint32_t *partials,
                        uint32_t *total_dev);

// Scratch for a radix sort or a digit pass over n keys: the tiles' digit
// counts (a tiles x RADIX_BINS matrix) and, after them, room for their scan
// out of place (one pass instead of three launches in place).
inline int64_t radix_hist_elems(int64_t n) {
    int64_t tiles = (n + RADIX_TILE - 1) / RADIX_TILE;
    return 2 * tiles * RADIX_BINS;
}

// Stable LSD sort of (key, value) pairs on key bits [0, bits), 8 bits per
// pass.  Ping-pongs between (k0, v0) and (k1, v1), all four n-element device
// buffers; *kout / *vout receive the buffers that hold the result.  With
// `iota` the incoming values are ignored and taken to be 0..n-1.  `hist`
// holds radix_hist_elems(n) entries, `partials` scan_scratch_elems of that.
template <typename K>
void radix_sort_pairs(Ctx &c, K *k0, uint32_t *v0, K *k1, uint32_t *v1, int64_t n, int bits, bool iota,
                      uint32_t *hist, uint32_t *partials, K **kout, uint32_t **vout);

// ------------------------------------------------------------------ chained prefixes
// Prefix sums across tiles in one pass (decoupled look-back): tile t
// publishes its own total, then the sum over every tile before it, in one
// 64-bit word (LB_INC: the low 32 bits are that inclusive prefix; LB_AGG:
// they are only the tile's own total; 0: nothing yet).  One warp of tile t
// reads the words of the 32 tiles before a point at once, adds the totals up
// to the nearest tile whose prefix is known, and moves 32 tiles further back
// only when none of the 32 has one.  Tiles take their index in the order
// their blocks start (from a counter), so every tile waited on has started
// and publishes its total without waiting on any other tile.  The wait is
// bounded all the same: after `spin_limit` polls the tile sums the input of
// every tile still silent itself (the scan is out of place, so that input is
// intact), sets ERR_TIMEOUT and goes on; its result stays exact.  Status
// words and the counter start at zero (one memset per pass).  With `fault`
// set every status word reads as silent, which makes the wait give up (the
// fault-injection test of the bound).
constexpr unsigned long long LB_AGG = 1ull << 62, LB_INC = 1ull << 63;
constexpr int64_t LB_SPIN_DEFAULT = 1 << 20;

// Called by all 32 lanes of one warp with the same arguments; returns the
// sum of `total` over the tiles before t (in every lane).  Tile q covers
// in[q * tile_elems, min((q + 1) * tile_elems, n)).
__device__ __forceinline__ uint32_t warp_lookback_exclusive(unsigned long long *status, int64_t t, uint32_t total,
                                                            const uint32_t *in, int64_t n, int64_t tile_elems,
                                                            int64_t spin_limit, bool fault, DevStatus *st) {
    const unsigned lane = lane_id();
    volatile unsigned long long *word = status;
    if (lane == 0) word[t] = (t == 0 ? LB_INC : LB_AGG) | total;
    if (t == 0) return 0;
    uint32_t excl = 0;
    int64_t j = t - 1;                       // lane i reads tile j - i
    int64_t spins = 0;
    bool gave_up = false;
    for (;;) {
        const int64_t q = j - (int64_t)lane;
        unsigned long long v = 0ull + LB_INC;                      // before tile 0: an empty known prefix
        if (q >= 0) v = fault ? 0ull : (unsigned long long)word[q];
        unsigned none = __ballot_sync(0xffffffffu, (v & (LB_INC | LB_AGG)) == 0);
        unsigned inc = __ballot_sync(0xffffffffu, (v & LB_INC) != 0);
        int first = inc ? __ffs(inc) - 1 : 32;                     // nearest tile with a known prefix
        unsigned upto = first == 32 ? 0xffffffffu : (2u << first) - 1u;
        if (none & upto) {                   // a tile on the way has published nothing yet
            if (!gave_up && ++spins <= spin_limit) {
                __nanosleep(64);
                continue;
            }
            gave_up = true;
            if ((none >> lane) & 1u) {       // its total, from its input
                const int64_t e = (q + 1) * tile_elems < n ? (q + 1) * tile_elems : n;
                uint32_t s = 0;
                for (int64_t i = q * tile_elems; i < e; ++i) s += in[i];
                v = LB_AGG | s;
            }
            inc = __ballot_sync(0xffffffffu, (v & LB_INC) != 0);
            first = inc ? __ffs(inc) - 1 : 32;
            upto = first == 32 ? 0xffffffffu : (2u << first) - 1u;
        }
        excl += warp_sum<uint32_t>(((upto >> lane) & 1u) ? (uint32_t)v : 0u);
        if (first < 32) break;
        j -= 32;
    }
    if (lane == 0) {
        if (gave_up) set_err(st, ERR_TIMEOUT);
        word[t] = LB_INC | (uint32_t)(excl + total);
    }
    return excl;
}

// ------------------------------------------------------------------ digit passes
// One stable counting pass whose 8-bit digit comes from a functor:
// digit(i) in [0, RADIX_BINS) for element i < n, or RADIX_BINS to leave the
// element out.  digit_offsets counts digits per tile of RADIX_TILE elements
// (digit-major matrix in `hist`, radix_hist_elems(n) entries) and scans the
// matrix; digit_rank then hands every counted element to epi(i, dest, digit),
// where dest is the position a stable sort by digit would give it, without
// moving anything itself.  epi returns problem bits; epi.done(bits) runs in every
// thread at the end (for warp votes).  Same tiles and ranking as the radix
// sort: warps own consecutive 512-element runs, ranked 32 at a time with
// peer groups from one ballot per digit bit.
template <typename DigitFn>
__global__ void __launch_bounds__(RADIX_THREADS) k_digit_hist(DigitFn digit, int64_t n, uint32_t *__restrict__ hist,
                                                              int64_t ntiles) {
    pdl_wait();
    __shared__ uint32_t h[RADIX_THREADS / 32][RADIX_BINS];
    const unsigned w = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) (&h[0][0])[i] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RADIX_TILE + w * (RADIX_TILE / 8);
#pragma unroll 4
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane_id();
        const unsigned d = i < n ? digit(i) : (unsigned)RADIX_BINS;
        if (d < RADIX_BINS) atomicAdd(&h[w][d], 1u);
    }
    __syncthreads();
    for (int d = threadIdx.x; d < RADIX_BINS; d += RADIX_THREADS) {
        uint32_t s = 0;
#pragma unroll
        for (int q = 0; q < RADIX_THREADS / 32; ++q) s += h[q][d];
        hist[(int64_t)d * ntiles + blockIdx.x] = s;
    }
}

template <typename DigitFn, typename Epi>
__global__ void __launch_bounds__(RADIX_THREADS) k_digit_rank(DigitFn digit, int64_t n,
                                                              const uint32_t *__restrict__ offs, int64_t ntiles,
                                                              Epi epi) {
    pdl_wait();
    __shared__ uint32_t wcnt[(RADIX_THREADS / 32) * RADIX_BINS];
    __shared__ uint32_t gbase[RADIX_BINS];
    const unsigned w = threadIdx.x >> 5, lane = lane_id();
    for (int i = threadIdx.x; i < (RADIX_THREADS / 32) * RADIX_BINS; i += RADIX_THREADS) wcnt[i] = 0;
    __syncthreads();
    const int64_t base = (int64_t)blockIdx.x * RADIX_TILE + w * (RADIX_TILE / 8);
    unsigned dig[RADIX_ITEMS];
    uint32_t rank[RADIX_ITEMS];
    const unsigned lt = lanemask_lt();
    unsigned peers[RADIX_ITEMS];
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {        // digits and peer groups first: independent
        const int64_t i = base + it * 32 + lane;
        const unsigned d = i < n ? digit(i) : (unsigned)RADIX_BINS;
        peers[it] = warp_peers8(d, d < RADIX_BINS);
        dig[it] = d;
    }
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const unsigned d = dig[it];
        const unsigned before = d < RADIX_BINS ? wcnt[w * RADIX_BINS + d] : 0u;
        __syncwarp();
        if (d < RADIX_BINS && (peers[it] & lt) == 0) wcnt[w * RADIX_BINS + d] = before + __popc(peers[it]);
        __syncwarp();
        rank[it] = before + __popc(peers[it] & lt);
    }
    __syncthreads();
    // RADIX_THREADS == RADIX_BINS: thread d turns digit d's per-warp counts
    // into exclusive prefixes and fetches the digit's global start
    {
        const unsigned d = threadIdx.x;
        uint32_t s = 0;
#pragma unroll
        for (int q = 0; q < RADIX_THREADS / 32; ++q) {
            const uint32_t x = wcnt[q * RADIX_BINS + d];
            wcnt[q * RADIX_BINS + d] = s;
            s += x;
        }
        gbase[d] = offs[(int64_t)d * ntiles + blockIdx.x];
    }
    __syncthreads();
    unsigned bits = 0;
#pragma unroll
    for (int it = 0; it < RADIX_ITEMS; ++it) {
        const int64_t i = base + it * 32 + lane;
        if (dig[it] < RADIX_BINS) bits |= epi(i, gbase[dig[it]] + wcnt[w * RADIX_BINS + dig[it]] + rank[it], dig[it]);
    }
    epi.done(bits);
}

// nbins: digits used (every digit below it); only those rows of the matrix
// are counted on and scanned.  The scan goes out of place, into the second
// half of `hist` (radix_hist_elems(n) entries: one pass); the offsets'
// address is returned for digit_rank.
template <typename DigitFn>
uint32_t *digit_offsets(Ctx &c, DigitFn digit, int64_t n, uint32_t *hist, uint32_t *partials,
                        int nbins = RADIX_BINS) {
    if (n <= 0) return hist;
    const int64_t ntiles = (n + RADIX_TILE - 1) / RADIX_TILE;
    launch(c, "digit_hist", k_digit_hist<DigitFn>, dim3((unsigned)ntiles), dim3(RADIX_THREADS), 0, digit, n, hist,
           ntiles);
    const int64_t m = ntiles * (int64_t)(nbins < 1 ? 1 : nbins);
    uint32_t *offs = hist + ntiles * RADIX_BINS;
    scan_exclusive_u32(c, hist, offs, m, partials, nullptr);
    return offs;
}

template <typename DigitFn, typename Epi>
void digit_rank(Ctx &c, const char *name, DigitFn digit, int64_t n, const uint32_t *hist, Epi epi) {
    if (n <= 0) return;
    const int64_t ntiles = (n + RADIX_TILE - 1) / RADIX_TILE;
    launch(c, name, k_digit_rank<DigitFn, Epi>, dim3((unsigned)ntiles), dim3(RADIX_THREADS), 0, digit, n, hist,
           ntiles, epi);
}

// Number of bits needed to represent v (0 for v == 0).
inline int bits_for(uint64_t v) {
    int b = 0;
    while (v) { b++; v >>= 1; }
    return b;
}

}  // namespace opattr
