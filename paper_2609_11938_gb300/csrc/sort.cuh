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

// Scratch for a scan of n elements: partial sums of the tiles (+1 for the total).
inline int64_t scan_scratch_elems(int64_t n) { return (n + SCAN_TILE - 1) / SCAN_TILE + 1; }

// out[i] = in[0] + ... + in[i-1]; *total_dev (device, may be NULL) = sum of all.
// in and out may alias.  `partials` holds scan_scratch_elems(n) u32.
void scan_exclusive_u32(Ctx &c, const uint32_t *in, uint32_t *out, int64_t n, uint32_t *partials,
                        uint32_t *total_dev);

// Scratch for a radix sort of n keys: histogram matrix + its scan partials.
inline int64_t radix_hist_elems(int64_t n) {
    int64_t tiles = (n + RADIX_TILE - 1) / RADIX_TILE;
    return tiles * RADIX_BINS;
}

// Stable LSD sort of (key, value) pairs on key bits [0, bits), 8 bits per
// pass.  Ping-pongs between (k0, v0) and (k1, v1), all four n-element device
// buffers; *kout / *vout receive the buffers that hold the result.  With
// `iota` the incoming values are ignored and taken to be 0..n-1.
template <typename K>
void radix_sort_pairs(Ctx &c, K *k0, uint32_t *v0, K *k1, uint32_t *v1, int64_t n, int bits, bool iota,
                      uint32_t *hist, uint32_t *partials, K **kout, uint32_t **vout);

// One stable counting pass on key bits [shift, shift + 8) that moves
// nothing: dest[i] receives the position element i would take.  hist /
// partials as for radix_sort_pairs.
template <typename K>
void radix_rank(Ctx &c, const K *keys, int64_t n, int shift, uint32_t *hist, uint32_t *partials, uint32_t *dest);

// Number of bits needed to represent v (0 for v == 0).
inline int bits_for(uint64_t v) {
    int b = 0;
    while (v) { b++; v >>= 1; }
    return b;
}

}  // namespace opattr
