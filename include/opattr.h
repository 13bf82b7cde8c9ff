/*
 * opattr.h -- C ABI of the GPU trace join behind hardware-attributed operator
 * profiling ("Hardware-Attributed Operator Profiling for PyTorch").
 *
 * The join has three calls, in this order (a fourth, opattr_attribute,
 * applies the attribution tiers of Fig. 2 between the first and the last):
 *   opattr_enclose   -- Algorithm 2 (Sec. 3.5): each kernel record gets the
 *                       innermost enclosing operator range on its stream.
 *   opattr_match     -- Algorithm 1 (Sec. 3.3): the i-th launch of a kernel
 *                       name pairs with the i-th Nsight Compute row of that
 *                       name; layer deduplication (Sec. 3.7) broadcasts a
 *                       representative layer's rows to its duplicates.
 *   opattr_aggregate -- Eq. (1) and Sec. 3.8.1: per-operator duration-weighted
 *                       means, sums and maxima of the 20-counter set
 *                       (Table 8), plus attributed / unattributed kernel time
 *                       (Fig. 4).
 *
 * Conventions shared by every call
 *  - Record and output arrays are DEVICE pointers owned by the caller, on the
 *    context's device.  Struct arguments themselves (and opattr_dedup's
 *    tables, the summaries and totals) live in HOST memory.
 *  - Work is ordered on the context's CUDA stream.  A call returns once its
 *    small host-side results have been copied back; the device outputs are
 *    then complete on that stream.  Inside a call, independent steps may run
 *    on a second stream the context owns, forked from and joined back into
 *    the caller's stream before the call returns.
 *  - Those small transfers (status block, level offsets, host-built tables)
 *    go through the device mapping of the context's pinned host buffers,
 *    moved by a small kernel of the library, not through the copy engines:
 *    a call does not wait behind bulk copies the caller has in flight on
 *    other streams (where the device cannot map them, cudaMemcpyAsync).
 *  - The library's kernels are programmatic dependent launches: each is
 *    scheduled as the kernel before it in the stream finishes, and waits,
 *    before touching memory, until that kernel has completed.  Work the
 *    caller queues on the stream before or after a call keeps its order.
 *  - Each call of the library is one NVTX range named after its entry point
 *    (visible on an Nsight Systems timeline).
 *  - n == 0 is valid everywhere and yields empty results.
 *  - Return value: negative = error (outputs undefined; the context stays
 *    usable except after OPATTR_E_CUDA, after which it must be destroyed),
 *    positive = warning (outputs valid), 0 = success.
 *  - Nothing is sorted in place; inputs are never written.
 */
#ifndef OPATTR_H
#define OPATTR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct opattr_ctx opattr_ctx;

typedef enum {
    OPATTR_OK = 0,
    OPATTR_W_COUNT_MISMATCH = 1,   /* some kernel name has different counts in the two traces */
    OPATTR_W_DEDUP_MISMATCH = 2,   /* some duplicate-layer kernel found no representative row */
    OPATTR_E_INVALID_ARG = -1,     /* bad pointer, size, id or value (see each call) */
    OPATTR_E_NOT_NESTED = -2,      /* ranges are not a laminar family per stream */
    OPATTR_E_DEPTH = -3,           /* a range depth is above 31 */
    OPATTR_E_COUNT_MISMATCH = -4,  /* count mismatch under OPATTR_MISMATCH_ERROR */
    OPATTR_E_CUDA = -5,            /* a CUDA call failed; destroy the context */
    OPATTR_E_OOM = -6,             /* device scratch could not be allocated */
    OPATTR_E_TIMEOUT = -7,         /* a bounded device-side wait gave up */
    OPATTR_E_STATE = -8            /* the context is unusable (after OPATTR_E_CUDA) */
} opattr_status;

/* What to do when a kernel name is launched a different number of times in
 * the Nsight Systems trace (replayed launches) and in the ncu rows. */
typedef enum {
    OPATTR_MISMATCH_SKIP_NAME = 0, /* every kernel of that name stays unmatched (Sec. 3.3 text) */
    OPATTR_MISMATCH_PREFIX = 1,    /* launch i takes row i while rows last (Algorithm 1 as printed) */
    OPATTR_MISMATCH_ERROR = 2      /* return OPATTR_E_COUNT_MISMATCH (limitations section) */
} opattr_mismatch_mode;

/* Range kinds are carried in op_id.  Algorithm 2 tests the range text: a
 * text without "::" (ProfilerStep#0, a layer or block marker) stops the walk;
 * a namespaced text that is not an operator (prims::, torch::) is skipped;
 * an operator (aten::, quantized::, a custom op) is collected.  Callers map
 * texts to these codes; every other op_id value names an operator. */
#define OPATTR_OP_STRUCTURAL 0xFFFFFFFFu
#define OPATTR_OP_NONOP 0xFFFFFFFEu
#define OPATTR_MAX_DEPTH 32
#define OPATTR_N_COUNTERS 20

/* Kernel records of the Nsight Systems trace (Sec. 3.1), one per launch.
 *   stream    u8[n]   stream the kernel ran on (< 256)
 *   start_ns  i64[n]  query point T: launch timestamp, ns (Sec. 3.5)
 *   dur_ns    i64[n]  kernel duration, ns, >= 0 (read by opattr_aggregate)
 *   name_id   u32[n]  kernel-name id (read by opattr_match)
 *   layer_id  i32[n]  layer partition tag, -1 outside layers, or NULL
 *                     (read by opattr_match when deduplication is on)
 * Time order of kernels is (start_ns, stream, array index).  No order is
 * required; records in time order take faster paths. */
typedef struct {
    const uint8_t *stream;
    const int64_t *start_ns;
    const int64_t *dur_ns;
    const uint32_t *name_id;
    const int32_t *layer_id;
    int64_t n;
} opattr_kernels;

/* NVTX ranges (Sec. 3.5), one per push/pop pair.
 *   stream    u8[n]   stream the range is keyed by
 *   start_ns, end_ns  i64[n]  closed interval [start, end], end >= start
 *   depth     u8[n]   nesting depth on its stream, 0 = outermost, <= 31
 *   op_id     u32[n]  operator id, or OPATTR_OP_STRUCTURAL / OPATTR_OP_NONOP
 * Per stream the ranges must be laminar: same-depth ranges overlap at most in
 * one instant (sorted by (start, end, index), each ends no later than the
 * next starts) and every range at depth d > 0 lies inside a depth d-1 range.
 * Violations return OPATTR_E_NOT_NESTED. */
typedef struct {
    const uint8_t *stream;
    const int64_t *start_ns;
    const int64_t *end_ns;
    const uint8_t *depth;
    const uint32_t *op_id;
    int64_t n;
} opattr_ranges;

/* Nsight Compute rows in launch order (Sec. 3.1).
 *   name_id   u32[n]       kernel-name id of the row
 *   counters  f32[n * 20]  row-major, counter #k (Table 8) at column k-1;
 *                          NaN = null (absent counter); values must be finite
 *                          or NaN; 16-byte aligned (read by opattr_aggregate)
 *   stream    u8[n]        stream of the row, or NULL.  Nsight Compute replays
 *                          one stream per run when a workload is multi-stream
 *                          (limitations paragraph of Sec. 5); with the rows of
 *                          those runs tagged here, opattr_match takes ordinals
 *                          per (name, stream) instead of per name, and name ids
 *                          must then be below 2^24.  Rows of one stream keep
 *                          their launch order; runs may come in any order. */
typedef struct {
    const uint32_t *name_id;
    const float *counters;
    int64_t n;
    const uint8_t *stream;
} opattr_ncu;

/* Layer deduplication tables (Sec. 3.7), HOST memory.
 *   class_of_layer  i32[n_layers]  equivalence class of each layer
 *   rep_of_class    i32[n_classes] representative layer of each class; it
 *                                  must belong to that class
 * Kernels of non-representative layers are not replayed: they take the row of
 * the representative's kernel at the same position within the layer (time
 * order), if that kernel has the same name and a row. */
typedef struct {
    const int32_t *class_of_layer;
    const int32_t *rep_of_class;
    int32_t n_layers;
    int32_t n_classes;
} opattr_dedup;

typedef struct {
    opattr_mismatch_mode mismatch; /* default OPATTR_MISMATCH_SKIP_NAME */
    int32_t dedup;                 /* 1: apply opattr_dedup when given (default 1) */
    int32_t checked;               /* reserved, 0 */
    int64_t spin_limit;            /* polls a device-side wait makes before it gives up (0 =
                                      default, 2^20; must be >= 0).  The only waits are those of
                                      the single-pass scans (a tile waiting for an earlier tile's
                                      prefix); one that gives up sums the earlier tiles' input
                                      itself, so results stay exact, and the call returns
                                      OPATTR_E_TIMEOUT */
} opattr_config;

/* Host-side result of opattr_match. */
typedef struct {
    int64_t kernels;               /* kernel records */
    int64_t replayed;              /* kernels with their own ncu row expected */
    int64_t direct;                /* kernels matched to a row directly */
    int64_t broadcast;             /* duplicate-layer kernels given a representative's row */
    int64_t unmatched;             /* kernels left without a row */
    int64_t names_mismatched;      /* names whose replayed and row counts differ */
    int64_t count_unmatched;       /* replayed kernels left unmatched by the count rule */
    int64_t dedup_mismatch;        /* duplicate-layer kernels without a usable source */
    int32_t fast_path;             /* 1: rows equal replayed kernels in time order */
    int32_t reserved;
} opattr_match_summary;

/* Device outputs of opattr_aggregate, one entry per op id, caller-allocated.
 *   kernel_count       i64[n_ops]       attributed kernels
 *   total_duration_ns  i64[n_ops]       sum of their durations
 *   matched_count      i64[n_ops]       attributed kernels that have a row
 *   agg                f64[20 * n_ops]  counter-major: agg[c * n_ops + op];
 *                                       NaN where no non-null value exists */
typedef struct {
    int64_t *kernel_count;
    int64_t *total_duration_ns;
    int64_t *matched_count;
    double *agg;
} opattr_op_aggregates;

/* Host-side totals of opattr_aggregate (Fig. 4 coverage). */
typedef struct {
    int64_t total_ns;              /* sum of all kernel durations */
    int64_t attributed_ns;         /* attributed kernels: range_of_kernel >= 0, or an operator */
    int64_t unattributed_ns;       /* total_ns - attributed_ns */
    int64_t kernels;
    int64_t attributed_kernels;
    int64_t matched_kernels;       /* attributed kernels with a row */
    double attributed_frac;        /* attributed_ns / total_ns, NaN if total_ns == 0 */
    double unattributed_frac;
} opattr_totals;

/* ---- Attribution tiers (Fig. 2, Sec. 3.4, Sec. 3.6) ----
 * Each kernel goes to the first tier that has an operator for it:
 *   HIGH      the torch.profiler correlation map (Sec. 3.4): an entry for the
 *             kernel's (name, invocation index), where the invocation index
 *             is the kernel's rank among all kernels of its name in time
 *             order (0 = first launch);
 *   NVTX      the innermost enclosing operator range (opattr_enclose);
 *   INDUCTOR  the Inductor fusion map (Sec. 3.6): an operator for the
 *             kernel's name;
 * and is unattributed otherwise.  The fusion map also enriches kernels of
 * the first two tiers: fused_with names the fused list's operator, and a
 * kernel is marked fused when its list holds several operators (or, for the
 * NVTX tier, when the walk collected several operator ranges). */
#define OPATTR_OP_NONE 0xFFFFFFFFu        /* no operator (same value as OPATTR_OP_STRUCTURAL) */
typedef enum {
    OPATTR_TIER_NONE = 0,
    OPATTR_TIER_HIGH = 1,
    OPATTR_TIER_NVTX = 2,
    OPATTR_TIER_INDUCTOR = 3
} opattr_tier;

/* torch.profiler correlation map (Phase 1 of the capture), device arrays in
 * any order:
 *   name_id     u32[n]  kernel-name id
 *   invocation  u32[n]  invocation index of that name
 *   op_id       u32[n]  operator the launch belongs to, < n_ops
 * A (name, invocation) pair that names an existing launch must appear once;
 * entries that name no launch (unknown name, index past the name's launch
 * count) are ignored. */
typedef struct {
    const uint32_t *name_id;
    const uint32_t *invocation;
    const uint32_t *op_id;
    int64_t n;
} opattr_corr;

/* Inductor fusion map (Sec. 3.6), device arrays indexed by kernel-name id:
 *   op_of_name  u32[n_names]  operator standing for the name's fused
 *                             operator list (< n_ops), or OPATTR_OP_NONE
 *   list_len    u8[n_names]   operators in that list (the "Original ATen"
 *                             comment), or NULL for 1
 * Names >= n_names have no entry. */
typedef struct {
    const uint32_t *op_of_name;
    const uint8_t *list_len;
    int64_t n_names;
} opattr_fusion;

/* Host-side result of opattr_attribute. */
typedef struct {
    int64_t kernels;
    int64_t high;                  /* kernels per tier */
    int64_t nvtx;
    int64_t inductor;
    int64_t none;
    int64_t fused;                 /* kernels marked fused */
    int64_t corr_used;             /* correlation entries that named a launch */
} opattr_attr_summary;

/* Create a context on `device` that orders its work on `cuda_stream` (a
 * cudaStream_t; NULL = the legacy default stream).  `cfg` may be NULL for
 * defaults.  The context owns reusable device scratch only.
 * Errors: OPATTR_E_INVALID_ARG (out NULL, bad device or mode),
 * OPATTR_E_CUDA. */
opattr_status opattr_create(opattr_ctx **out, int device, void *cuda_stream, const opattr_config *cfg);

/* Algorithm 2 for every kernel: range_of_kernel[k] = index of the innermost
 * operator range enclosing kernel k, or -1; n_op_enclosing[k] = number of
 * operator ranges collected by the walk (is_fused = value > 1).
 * Per depth d the representative is the greatest (start, end, index) among
 * depth-d ranges of the kernel's stream with start <= T <= end; the walk goes
 * from the deepest representative outward, collects operators, skips
 * OPATTR_OP_NONOP, stops at OPATTR_OP_STRUCTURAL.
 * Reads kernels->stream, start_ns and all range fields.
 *   range_of_kernel  i32[kernels->n]  device, required
 *   n_op_enclosing   u8[kernels->n]   device, may be NULL
 * Errors: OPATTR_E_INVALID_ARG (NULL arrays with n > 0, end < start, more
 * than 2^30 ranges), OPATTR_E_DEPTH, OPATTR_E_NOT_NESTED, OPATTR_E_OOM,
 * OPATTR_E_CUDA. */
opattr_status opattr_enclose(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                             int32_t *range_of_kernel, uint8_t *n_op_enclosing);

/* Algorithm 1 with the context's mismatch mode.  ncu_idx_of_kernel[k] = ncu
 * row of kernel k or -1; match_kind[k] = 0 none, 1 direct, 2 broadcast.
 * Ordinals are taken over replayed kernels in time order and over rows in
 * array order, per name -- or per (name, stream) when ncu->stream is given:
 * then a kernel's "name" in counts, ordinals and mismatch modes is the pair,
 * while the duplicate-layer check of Sec. 3.7 still compares plain names (a
 * class's representative layer may run on another stream).  When the two
 * sides, each partitioned stably by stream, carry the same keys position by
 * position, the pairing is read off directly.  `dedup` (host) may be NULL;
 * deduplication also needs kernels->layer_id and cfg.dedup = 1.
 * Reads kernels->stream, start_ns, name_id (and layer_id), ncu->name_id (and
 * ncu->stream).
 *   ncu_idx_of_kernel  i32[kernels->n]  device, required
 *   match_kind         u8[kernels->n]   device, may be NULL
 *   host_summary       host, may be NULL
 * Returns OPATTR_W_COUNT_MISMATCH (skip-name: some name mismatched; prefix:
 * some kernel found no row), else OPATTR_W_DEDUP_MISMATCH when a duplicate
 * found no source.  Errors: OPATTR_E_INVALID_ARG (layer id >= n_layers, bad
 * tables, a name id >= 2^24 with ncu->stream), OPATTR_E_COUNT_MISMATCH (error
 * mode), OPATTR_E_OOM, OPATTR_E_CUDA. */
opattr_status opattr_match(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ncu *ncu,
                           const opattr_dedup *dedup, int32_t *ncu_idx_of_kernel, uint8_t *match_kind,
                           opattr_match_summary *host_summary);

/* Eq. (1) per operator: for op = op_id[range_of_kernel[k]], counts and
 * duration sums in int64 (exact); per counter, over attributed kernels with a
 * row and a non-null value: SUM of values, MAX of values, or the
 * duration-weighted mean sum(m*d)/sum(d) (Table 8 picks which); NaN for an
 * empty set or a zero total weight.  Floating-point results are within 1e-9
 * relative of an fp64 evaluation (float-float accumulation, see the design
 * notes).  Every op id in [0, n_ops) is written.
 * Reads kernels->dur_ns, ranges->op_id, ncu->counters.
 *   range_of_kernel    i32[kernels->n]  device, values in [-1, ranges->n);
 *                                       or NULL: then ranges->op_id holds
 *                                       one operator per kernel
 *                                       (ranges->n == kernels->n), and
 *                                       OPATTR_OP_NONE marks unattributed
 *                                       kernels (opattr_attribute's output)
 *   ncu_idx_of_kernel  i32[kernels->n]  device, values in [-1, ncu->n)
 *   dev_out            host struct of device pointers, see above
 *   host_totals        host, may be NULL
 * Errors: OPATTR_E_INVALID_ARG (index out of range, attributed range that is
 * not an operator below n_ops, an operator >= n_ops other than
 * OPATTR_OP_NONE, negative duration, infinite counter, counters not 16-byte
 * aligned),
 * OPATTR_E_OOM, OPATTR_E_CUDA. */
opattr_status opattr_aggregate(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                               const int32_t *range_of_kernel, const opattr_ncu *ncu,
                               const int32_t *ncu_idx_of_kernel, uint32_t n_ops,
                               const opattr_op_aggregates *dev_out, opattr_totals *host_totals);

/* The whole join in one call: opattr_enclose, opattr_match and
 * opattr_aggregate on the same kernel records, in that order, with the same
 * arguments and outputs as the three calls (range_of_kernel is written by the
 * enclosure and read by the aggregation, ncu_idx_of_kernel likewise from the
 * matching).  The kernel records' time order is verified once for both the
 * enclosure and the matching.  With as many ncu rows as kernels (no
 * deduplication, no per-stream rows), the identity pairing of the matching
 * runs beside the enclosure and, when the kernels are in time order, the
 * enclosure's verdict is read with the aggregation's status: the outputs are
 * those of the three calls all the same (a disagreeing name redoes the
 * matching and the aggregation; ranges that need the enclosure's fully
 * sorted pass run the join again).
 *   n_op_enclosing, match_kind, host_summary, host_totals  may be NULL
 * Returns the first error of the three steps in step order (an error of the
 * enclosure is returned even when the aggregation already ran), else the
 * matching's warning if it gave one, else OPATTR_OK. */
opattr_status opattr_join(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                          const opattr_ncu *ncu, const opattr_dedup *dedup, uint32_t n_ops,
                          int32_t *range_of_kernel, uint8_t *n_op_enclosing, int32_t *ncu_idx_of_kernel,
                          uint8_t *match_kind, const opattr_op_aggregates *dev_out,
                          opattr_match_summary *host_summary, opattr_totals *host_totals);

/* The attribution tiers of Fig. 2 for every kernel (see above).
 *   range_of_kernel  i32[kernels->n]  device, opattr_enclose's result
 *   n_op_enclosing   u8[kernels->n]   device, opattr_enclose's count, or NULL
 *   corr             host struct of device arrays, or NULL (no HIGH tier)
 *   fusion           host struct of device arrays, or NULL (no INDUCTOR tier)
 *   op_of_kernel     u32[kernels->n]  device, required: the kernel's operator
 *                                     or OPATTR_OP_NONE
 *   tier             u8[kernels->n]   device, may be NULL: opattr_tier
 *   fused_with       u32[kernels->n]  device, may be NULL: the fusion map's
 *                                     operator for the kernel's name, or
 *                                     OPATTR_OP_NONE
 *   is_fused         u8[kernels->n]   device, may be NULL: 1 if the kernel's
 *                                     fused list has several operators, or
 *                                     (NVTX tier) n_op_enclosing > 1
 *   host_summary     host, may be NULL
 * Reads kernels->stream, start_ns, name_id and ranges->op_id.  op_of_kernel
 * feeds opattr_aggregate with range_of_kernel NULL.
 * Errors: OPATTR_E_INVALID_ARG (range index out of [-1, ranges->n), an NVTX
 * range that is not an operator below n_ops, a correlation or fusion
 * operator >= n_ops, a repeated (name, invocation) pair that names a
 * launch), OPATTR_E_OOM, OPATTR_E_CUDA. */
opattr_status opattr_attribute(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                               const int32_t *range_of_kernel, const uint8_t *n_op_enclosing, const opattr_corr *corr,
                               const opattr_fusion *fusion, uint32_t n_ops, uint32_t *op_of_kernel, uint8_t *tier,
                               uint32_t *fused_with, uint8_t *is_fused, opattr_attr_summary *host_summary);

/* Class roll-up: the records of opattr_aggregate per operator class instead
 * of per operator (the per-class breakdowns of the case studies, where every
 * dispatch aten::mm_N counts towards aten::mm).  class_of_op maps each op id
 * to a class below n_classes, or OPATTR_OP_NONE to leave the op out.  Per
 * class: kernel count, duration, matched count and the 20 counters by Table
 * 8's rules over all kernels of the class's operators -- Eq. (1) at class
 * granularity, so a class's duration-weighted mean weighs every kernel, not
 * every operator.  Every class in [0, n_classes) is written (empty classes
 * get zero counts and NaN counters).
 *   kernels, ranges, range_of_kernel, ncu, ncu_idx_of_kernel, n_ops: as for
 *                      opattr_aggregate (range_of_kernel may be NULL there too)
 *   class_of_op        u32[n_ops]  device
 *   dev_out            host struct of device pointers, n_classes entries
 * Errors: OPATTR_E_INVALID_ARG (as opattr_aggregate, a class >= n_classes
 * other than OPATTR_OP_NONE, n_classes > 2^24), OPATTR_E_OOM, OPATTR_E_CUDA. */
opattr_status opattr_rollup(opattr_ctx *ctx, const opattr_kernels *kernels, const opattr_ranges *ranges,
                            const int32_t *range_of_kernel, const opattr_ncu *ncu, const int32_t *ncu_idx_of_kernel,
                            uint32_t n_ops, const uint32_t *class_of_op, uint32_t n_classes,
                            const opattr_op_aggregates *dev_out);

/* ---- profile.json (App. A.4 schema) ----
 * A host-side writer over the join's outputs: one entry per attributed
 * operator with its kernels (name, attribution tier and confidence,
 * duration, stream, the 20 raw counters of its ncu row) and its aggregated
 * record, then the unattributed kernels.  Counter fields carry the profile
 * names of Table 8; NaN is written as null.  Every array here is HOST memory
 * (copy the device outputs back first). */
typedef struct {
    const char *model_name;            /* capture_metadata fields, NULL = omitted */
    const char *device_name;
    const char *compile_mode;
    const char *capture_timestamp_utc;
    int32_t include_kernels;           /* 0: operators without per-kernel records (large traces) */
} opattr_profile_meta;

typedef struct {
    const char *const *kernel_name;    /* [n_kernel_names] by name id, NULL = "kernel_<id>" */
    int64_t n_kernel_names;
    const char *const *op_name;        /* [n_ops] canonical operator name (aten::mm), NULL = "op_<id>" */
    const int64_t *op_call_index;      /* [n_ops] dispatch ordinal (operator_id = name_index), NULL = op id */
} opattr_profile_names;

/* Writes the document to `path`.
 *   kernels          host struct of HOST arrays: stream, dur_ns, name_id, n
 *   op_of_kernel     u32[kernels->n]  operator of each kernel or OPATTR_OP_NONE
 *   tier             u8[kernels->n]   opattr_tier, or NULL (NVTX for attributed kernels)
 *   is_fused         u8[kernels->n]   or NULL
 *   fused_with       u32[kernels->n]  or NULL (operator of the kernel's fused list)
 *   ncu_idx_of_kernel i32[kernels->n] row of each kernel or -1
 *   counters         f32[n_rows * 20] the ncu rows
 *   ops              host struct of HOST arrays, n_ops entries (opattr_aggregate's output)
 *   bytes_written    may be NULL
 * Errors: OPATTR_E_INVALID_ARG (NULL required array, an operator >= n_ops,
 * a row index out of range, the file cannot be written). */
opattr_status opattr_write_profile(const char *path, const opattr_profile_meta *meta,
                                   const opattr_profile_names *names, const opattr_kernels *kernels,
                                   const uint32_t *op_of_kernel, const uint8_t *tier, const uint8_t *is_fused,
                                   const uint32_t *fused_with, const int32_t *ncu_idx_of_kernel, const float *counters,
                                   int64_t n_rows, uint32_t n_ops, const opattr_op_aggregates *ops,
                                   int64_t *bytes_written);

/* Free the context and its scratch.  NULL is ignored. */
void opattr_destroy(opattr_ctx *ctx);

/* Static string for a status code. */
const char *opattr_status_string(opattr_status status);

/* Launch accounting and per-kernel timing.  With timing on, every kernel
 * launch of the context is bracketed by CUDA events on the context's stream
 * and its duration accumulated per kernel name.  opattr_timing_report fills
 * up to `cap` entries (names are static strings) and returns how many kernel
 * names have been seen; opattr_launch_count returns the number of kernels the
 * context has launched since creation or the last reset. */
opattr_status opattr_set_timing(opattr_ctx *ctx, int enable);
/* With timing on, bracket only the launches of the kernel named `kernel` (a
 * name opattr_timing_report lists); NULL brackets every launch again.  The
 * name is copied. */
opattr_status opattr_set_timing_only(opattr_ctx *ctx, const char *kernel);
int opattr_timing_report(opattr_ctx *ctx, const char **names, double *total_ms, int64_t *launches, int cap);
void opattr_timing_reset(opattr_ctx *ctx);
int64_t opattr_launch_count(const opattr_ctx *ctx);

/* No-allocation variant of opattr_match.  The paper has no counterpart: it
 * exists for callers that cannot allocate device memory -- an attribution
 * pass running inside the profiled application (an injection library or a
 * profiler callback) must leave that application's device memory untouched,
 * and some hosts own all device memory through a caching allocator or forbid
 * allocation on a hot path.
 *   Same inputs, outputs, ordering and status codes as opattr_match with
 *   layer deduplication off, on the stream `cuda_stream` of the current
 *   device, with `mismatch` in place of the context's mode.  No context.
 *   All scratch (6 MB) lives in one fixed device array inside the library;
 *   every GPU that loads the library holds it until exit.  It holds the
 *   general (sorting) path at the limit below.
 *   kernels->n and ncu->n must each be at most OPATTR_MATCH_NOALLOC_MAX,
 *   else OPATTR_E_INVALID_ARG; per-stream ordinals are not available here
 *   (ncu->stream must be NULL, else OPATTR_E_INVALID_ARG).
 *   Every call looks up the array's device address in the CUDA context
 *   current at the call (a host-side lookup), so a device reset or another
 *   context between calls is safe.  The first call in a context may also load
 *   the library's device code (lazy module loading), and that is when the
 *   array itself comes into being: make one warm-up call per device and
 *   context outside any region that must not allocate, and before any stream
 *   capture.  The call synchronises its stream and copies to host memory, so
 *   it cannot be captured into a CUDA graph.
 *   Calls share the array.  Host threads are serialised inside the call, and
 *   each call, whatever it returns, finishes its device work before it
 *   returns; a caller that lets other work on the GPU touch the same memory
 *   concurrently races.
 *   Allocates nothing after that first call: no cudaMalloc, cudaFree or
 *   pinned host memory. */
#define OPATTR_MATCH_NOALLOC_MAX 65536
opattr_status opattr_match_noalloc(const opattr_kernels *kernels, const opattr_ncu *ncu,
                                   opattr_mismatch_mode mismatch, int32_t *ncu_idx_of_kernel, uint8_t *match_kind,
                                   opattr_match_summary *host_summary, void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* OPATTR_H */
