// util.cuh -- steps shared by the three calls: kernel time-order check and
// time-order permutation.
#pragma once
#include "common.cuh"
#include "sort.cuh"

namespace opattr {

// Sets F_K_UNSORTED unless (start_ns, stream) is non-decreasing along the
// array, and records min / max start in MM_KSTART_MIN / MM_KSTART_MAX.  With
// stream_hist (256 zeroed counters), also counts the kernels of each stream;
// with tile_hist (radix_hist_elems(n) counters), writes the stream counts of
// every RADIX_TILE tile of the array as a stream-major matrix.
void check_kernel_order(Ctx &c, const uint8_t *stream, const int64_t *start, int64_t n,
                        uint32_t *stream_hist = nullptr, uint32_t *tile_hist = nullptr);

// Scratch (bytes) of kernel_time_order for n kernels.
size_t kernel_order_scratch(int64_t n);

// Permutation of kernel indices into time order (start, stream, index) by a
// stable radix sort of ((start - min_start) << sbits | stream).  Needs the
// min / max from check_kernel_order in c.h_status.  With scmap (device,
// [256]: increasing compact ids of the streams that have kernels) the key
// holds the compact id in stream_bits bits instead of the id in 8, which
// saves a pass when the span and the stream count allow.  Returns a device
// array of n indices carved from `a`, or NULL on arena exhaustion.
uint32_t *kernel_time_order(Ctx &c, struct Arena &a, const uint8_t *stream, const int64_t *start, int64_t n,
                            const uint8_t *scmap = nullptr, int stream_bits = 8);

}  // namespace opattr
