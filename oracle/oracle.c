/*
 * oracle.c -- plain, slow CPU reference for the attribution join.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test-suite, the smoke check and the
 * benchmark's CPU-baseline leg load this file.  The CUDA library never calls,
 * links or includes it, and this file includes nothing of the library's.
 *
 * What it computes (paper: "Hardware-Attributed Operator Profiling for
 * PyTorch"):
 *   enclosure    -- Algorithm 2 (NVTX enclosure attribution, Sec. 3.5):
 *                   innermost enclosing operator range per kernel on the
 *                   kernel's stream, walk from innermost to outermost,
 *                   collect operator ranges, stop at a range without a
 *                   namespace, skip other namespaced ranges; is_fused when
 *                   more than one operator range is collected.
 *   matching     -- Algorithm 1 (invocation-order matching, Sec. 3.3): the
 *                   i-th launch of a kernel name pairs with the i-th ncu row
 *                   of that name; count validation before assignment; layer
 *                   deduplication (Sec. 3.7): skipped duplicates inherit the
 *                   counters of their class representative by position.
 *   aggregation  -- Eq. (1) duration-weighted mean, plain sum for additive
 *                   counters, maximum for per-kernel constants (Sec. 3.8.1),
 *                   per counter as Table 8 assigns; total/attributed/
 *                   unattributed kernel time (Sec. 3.2 durations, Fig. 4).
 *
 * Readings taken where the paper is silent (the same list is kept with the
 * design notes):
 *   - ranges and kernels are keyed by stream; the query point T of a kernel is
 *     its start timestamp (one clock domain in the synthetic traces);
 *   - closed intervals s <= T <= e;
 *   - one representative per depth: among the depth-d ranges on the stream
 *     that contain T, the greatest (start, end, index); the chain visited by
 *     the walk is those representatives from the deepest depth up;
 *   - op ids encode the range text: OP_STRUCTURAL (no "::") stops the walk,
 *     OP_NONOP (namespaced, not an operator) is skipped, any other value is an
 *     operator;
 *   - kernel time order is (start, stream, input index); ncu rows are in
 *     launch order;
 *   - count mismatch: three modes -- skip the whole name (Sec. 3.3 text),
 *     prefix assignment with a warning (Algorithm 1 as printed), or raise
 *     (limitations section);
 *   - dedup position = rank among the kernels tagged with the same layer, in
 *     time order; the representative's kernel at that position must carry the
 *     same name;
 *   - NaN counters are null and take no part in SUM, MAX or DW; an empty set
 *     or a zero weight gives NaN; infinite counters are rejected.
 *
 * Floating point: fp64 throughout, sums with Neumaier's compensated summation
 * (Neumaier 1974), serially in kernel index order.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#define ORC_OK 0
#define ORC_W_COUNT_MISMATCH 1
#define ORC_W_DEDUP_MISMATCH 2
#define ORC_E_INVALID_ARG (-1)
#define ORC_E_NOT_NESTED (-2)
#define ORC_E_DEPTH (-3)
#define ORC_E_COUNT_MISMATCH (-4)
#define ORC_E_OOM (-6)

#define OP_STRUCTURAL 0xFFFFFFFFu
#define OP_NONOP 0xFFFFFFFEu
#define MAX_DEPTH 32
#define NC 20

enum { MODE_SKIP_NAME = 0, MODE_PREFIX = 1, MODE_ERROR = 2 };
enum { AGG_SUM = 0, AGG_DW = 1, AGG_MAX = 2 };

/* Table 8: aggregation rule of counters #1..#20 (index = number - 1). */
static const int AGG_RULE[NC] = {
    AGG_SUM, AGG_SUM, AGG_SUM,                  /* 1 gpu time, 2 dram read, 3 dram written */
    AGG_DW, AGG_DW, AGG_DW, AGG_DW, AGG_DW,     /* 4 mem thr, 5 dram thr, 6 mem busy, 7 L1 hit, 8 L2 hit */
    AGG_DW, AGG_DW,                             /* 9 sm thr, 10 tensor active */
    AGG_SUM,                                    /* 11 sm active cycles */
    AGG_DW, AGG_DW, AGG_DW,                     /* 12 occupancy, 13 warp cycles/instr, 14 eligible */
    AGG_SUM,                                    /* 15 executed instructions */
    AGG_DW, AGG_DW,                             /* 16 ipc, 17 threads/warp */
    AGG_MAX,                                    /* 18 registers/thread */
    AGG_SUM,                                    /* 19 local spills */
    AGG_MAX,                                    /* 20 dynamic smem/block */
};

int orc_agg_rule(int c) { return (c >= 0 && c < NC) ? AGG_RULE[c] : -1; }

/* ------------------------------------------------------------------ sorting */
/* A plain stable merge sort of an index array under a comparison callback. */
typedef int (*cmp_fn)(int64_t a, int64_t b, const void *ctx);

static void msort_rec(int64_t *a, int64_t *tmp, int64_t n, cmp_fn cmp, const void *ctx) {
    if (n < 2) return;
    int64_t h = n / 2;
    msort_rec(a, tmp, h, cmp, ctx);
    msort_rec(a + h, tmp, n - h, cmp, ctx);
    int64_t i = 0, j = h, o = 0;
    while (i < h && j < n) tmp[o++] = (cmp(a[j], a[i], ctx) < 0) ? a[j++] : a[i++];
    while (i < h) tmp[o++] = a[i++];
    while (j < n) tmp[o++] = a[j++];
    memcpy(a, tmp, sizeof(int64_t) * n);
}
static int stable_sort_idx(int64_t *a, int64_t n, cmp_fn cmp, const void *ctx) {
    int64_t *tmp = (int64_t *)malloc(sizeof(int64_t) * (n ? n : 1));
    if (!tmp) return ORC_E_OOM;
    msort_rec(a, tmp, n, cmp, ctx);
    free(tmp);
    return ORC_OK;
}

/* ------------------------------------------------------------------ ranges */
typedef struct {
    int64_t R;
    const uint8_t *stream, *depth;
    const int64_t *start, *end;
    const uint32_t *op;
} ranges_t;

/* (stream, depth, start, end, index) ascending */
static int cmp_level_order(int64_t a, int64_t b, const void *ctx) {
    const ranges_t *r = (const ranges_t *)ctx;
    if (r->stream[a] != r->stream[b]) return r->stream[a] < r->stream[b] ? -1 : 1;
    if (r->depth[a] != r->depth[b]) return r->depth[a] < r->depth[b] ? -1 : 1;
    if (r->start[a] != r->start[b]) return r->start[a] < r->start[b] ? -1 : 1;
    if (r->end[a] != r->end[b]) return r->end[a] < r->end[b] ? -1 : 1;
    return a < b ? -1 : (a > b);
}

/* Is range a "greater" representative than b: (start, end, index) order. */
static int rep_greater(const ranges_t *r, int64_t a, int64_t b) {
    if (r->start[a] != r->start[b]) return r->start[a] > r->start[b];
    if (r->end[a] != r->end[b]) return r->end[a] > r->end[b];
    return a > b;
}

/* Argument checks shared by both modes: end >= start, then depth <= 31. */
static int check_range_fields(const ranges_t *r) {
    for (int64_t i = 0; i < r->R; ++i)
        if (r->end[i] < r->start[i]) return ORC_E_INVALID_ARG;
    for (int64_t i = 0; i < r->R; ++i)
        if (r->depth[i] >= MAX_DEPTH) return ORC_E_DEPTH;
    return ORC_OK;
}

/* Laminar-family check written straight from its definition, O(R^2):
 *  (1) two ranges on the same stream and depth overlap at most in one
 *      instant: the one first in (start, end, index) order ends no later than
 *      the other starts;
 *  (2) a range at depth d > 0 lies inside some depth d-1 range of its stream.
 * Ranges come from push/pop pairs (Sec. 3.5), so both hold for real traces. */
int orc_validate_ranges_brute(int64_t R, const uint8_t *stream, const int64_t *start, const int64_t *end,
                              const uint8_t *depth) {
    ranges_t r = { R, stream, depth, start, end, NULL };
    int st = check_range_fields(&r);
    if (st) return st;
    for (int64_t a = 0; a < R; ++a) {
        int has_parent = depth[a] == 0;
        for (int64_t b = 0; b < R; ++b) {
            if (b == a || stream[b] != stream[a]) continue;
            if (depth[b] == depth[a]) {
                int64_t first = rep_greater(&r, a, b) ? b : a, second = first == a ? b : a;
                if (end[first] > start[second]) return ORC_E_NOT_NESTED;
            } else if (depth[b] + 1 == depth[a] && start[b] <= start[a] && end[a] <= end[b]) {
                has_parent = 1;
            }
        }
        if (!has_parent) return ORC_E_NOT_NESTED;
    }
    return ORC_OK;
}

/* The same checks through sorted level lists: adjacent pairs of a level in
 * (start, end, index) order, and for every range a search of the parent level
 * for the greatest range starting at or before it. */
typedef struct {
    int64_t *ord;                  /* range indices in (stream, depth, start, end, index) order */
    int64_t *lvl_off;              /* 256 * 32 + 1 offsets into ord */
} levels_t;

static int build_levels(const ranges_t *r, levels_t *L) {
    L->ord = (int64_t *)malloc(sizeof(int64_t) * (r->R ? r->R : 1));
    L->lvl_off = (int64_t *)calloc(256 * MAX_DEPTH + 1, sizeof(int64_t));
    if (!L->ord || !L->lvl_off) return ORC_E_OOM;
    for (int64_t i = 0; i < r->R; ++i) L->ord[i] = i;
    int st = stable_sort_idx(L->ord, r->R, cmp_level_order, r);
    if (st) return st;
    for (int64_t i = 0; i < r->R; ++i) L->lvl_off[r->stream[i] * MAX_DEPTH + r->depth[i] + 1]++;
    for (int l = 0; l < 256 * MAX_DEPTH; ++l) L->lvl_off[l + 1] += L->lvl_off[l];
    return ORC_OK;
}
static void free_levels(levels_t *L) { free(L->ord); free(L->lvl_off); }

/* Last position p in level (s, d) with start <= T, or -1. */
static int64_t level_last_start_le(const ranges_t *r, const levels_t *L, int s, int d, int64_t T) {
    int64_t lo = L->lvl_off[s * MAX_DEPTH + d], hi = L->lvl_off[s * MAX_DEPTH + d + 1];
    int64_t a = lo, b = hi;        /* first position with start > T */
    while (a < b) {
        int64_t m = a + (b - a) / 2;
        if (r->start[L->ord[m]] <= T) a = m + 1; else b = m;
    }
    return a > lo ? a - 1 : -1;
}

static int validate_levels(const ranges_t *r, const levels_t *L) {
    for (int l = 0; l < 256 * MAX_DEPTH; ++l) {
        for (int64_t p = L->lvl_off[l]; p + 1 < L->lvl_off[l + 1]; ++p)
            if (r->end[L->ord[p]] > r->start[L->ord[p + 1]]) return ORC_E_NOT_NESTED;
    }
    for (int64_t i = 0; i < r->R; ++i) {
        if (r->depth[i] == 0) continue;
        int64_t p = level_last_start_le(r, L, r->stream[i], r->depth[i] - 1, r->start[i]);
        if (p < 0 || r->end[L->ord[p]] < r->end[i]) return ORC_E_NOT_NESTED;
    }
    return ORC_OK;
}

int orc_validate_ranges_indexed(int64_t R, const uint8_t *stream, const int64_t *start, const int64_t *end,
                                const uint8_t *depth) {
    ranges_t r = { R, stream, depth, start, end, NULL };
    int st = check_range_fields(&r);
    if (st) return st;
    levels_t L;
    st = build_levels(&r, &L);
    if (!st) st = validate_levels(&r, &L);
    free_levels(&L);
    return st;
}

/* Algorithm 2 walk over the representative chain, deepest first.
 * chain[d] = range index of the depth-d representative, or -1. */
static void walk_chain(const ranges_t *r, const int64_t *chain, int32_t *out_range, uint8_t *out_nop) {
    int32_t first = -1;
    int n_op = 0;
    for (int d = MAX_DEPTH - 1; d >= 0; --d) {
        int64_t x = chain[d];
        if (x < 0) continue;
        uint32_t op = r->op[x];
        if (op == OP_STRUCTURAL) break;            /* no "::" in the text: structural boundary */
        if (op == OP_NONOP) continue;              /* namespaced but not an operator: skip */
        if (first < 0) first = (int32_t)x;         /* innermost attributed range */
        n_op++;
    }
    *out_range = first;
    *out_nop = (uint8_t)n_op;
}

/* Enclosure, brute force: every range of the kernel's stream is tested.
 * mode 0 = brute, 1 = indexed (level lists + binary search), 2 = the brute
 * chain after the indexed laminar check (the all-pairs check is quadratic in
 * the ranges; this mode serves kernel samples of traces with millions of
 * ranges, whose validity the indexed check, itself pinned against the
 * all-pairs one, decides). */
int orc_enclose(int mode, int64_t K, const uint8_t *k_stream, const int64_t *k_start,
                int64_t R, const uint8_t *r_stream, const int64_t *r_start, const int64_t *r_end,
                const uint8_t *r_depth, const uint32_t *r_op, int32_t *out_range, uint8_t *out_nop) {
    ranges_t r = { R, r_stream, r_depth, r_start, r_end, r_op };
    int st = mode == 0 ? orc_validate_ranges_brute(R, r_stream, r_start, r_end, r_depth)
                       : orc_validate_ranges_indexed(R, r_stream, r_start, r_end, r_depth);
    if (st) return st;
    int64_t chain[MAX_DEPTH];
    if (mode == 0 || mode == 2) {
        /* per-stream lists of range indices, so the scan visits one stream */
        int64_t *cnt = (int64_t *)calloc(257, sizeof(int64_t));
        int64_t *lst = (int64_t *)malloc(sizeof(int64_t) * (R ? R : 1));
        if (!cnt || !lst) { free(cnt); free(lst); return ORC_E_OOM; }
        for (int64_t i = 0; i < R; ++i) cnt[r_stream[i] + 1]++;
        for (int s = 0; s < 256; ++s) cnt[s + 1] += cnt[s];
        int64_t fill[256];
        for (int s = 0; s < 256; ++s) fill[s] = cnt[s];
        for (int64_t i = 0; i < R; ++i) lst[fill[r_stream[i]]++] = i;
        for (int64_t k = 0; k < K; ++k) {
            int s = k_stream[k];
            int64_t T = k_start[k];
            for (int d = 0; d < MAX_DEPTH; ++d) chain[d] = -1;
            for (int64_t q = cnt[s]; q < cnt[s + 1]; ++q) {
                int64_t i = lst[q];
                if (r_start[i] <= T && T <= r_end[i]) {           /* closed interval */
                    int d = r_depth[i];
                    if (chain[d] < 0 || rep_greater(&r, i, chain[d])) chain[d] = i;
                }
            }
            walk_chain(&r, chain, &out_range[k], &out_nop[k]);
        }
        free(cnt); free(lst);
        return ORC_OK;
    }
    levels_t L;
    st = build_levels(&r, &L);
    if (st) { free_levels(&L); return st; }
    for (int64_t k = 0; k < K; ++k) {
        int s = k_stream[k];
        int64_t T = k_start[k];
        for (int d = 0; d < MAX_DEPTH; ++d) {
            int64_t p = level_last_start_le(&r, &L, s, d, T);
            chain[d] = (p >= 0 && r_end[L.ord[p]] >= T) ? L.ord[p] : -1;
        }
        walk_chain(&r, chain, &out_range[k], &out_nop[k]);
    }
    free_levels(&L);
    return ORC_OK;
}

/* ------------------------------------------------------------------ matching */
typedef struct { const int64_t *start; const uint8_t *stream; } korder_t;
static int cmp_time(int64_t a, int64_t b, const void *ctx) {
    const korder_t *o = (const korder_t *)ctx;
    if (o->start[a] != o->start[b]) return o->start[a] < o->start[b] ? -1 : 1;
    if (o->stream[a] != o->stream[b]) return o->stream[a] < o->stream[b] ? -1 : 1;
    return a < b ? -1 : (a > b);
}
typedef struct { const uint32_t *key; } ukey_t;
static int cmp_u32key(int64_t a, int64_t b, const void *ctx) {
    const ukey_t *u = (const ukey_t *)ctx;
    if (u->key[a] != u->key[b]) return u->key[a] < u->key[b] ? -1 : 1;
    return 0;                      /* stable sort keeps the incoming order */
}

/* Distinct-name dictionary: sorted unique names + lookup by binary search. */
typedef struct { uint32_t *name; int64_t n; } dict_t;
static int dict_build(dict_t *D, const uint32_t *a, int64_t na, const uint32_t *b, int64_t nb) {
    int64_t n = na + nb;
    uint32_t *v = (uint32_t *)malloc(sizeof(uint32_t) * (n ? n : 1));
    int64_t *ix = (int64_t *)malloc(sizeof(int64_t) * (n ? n : 1));
    D->name = (uint32_t *)malloc(sizeof(uint32_t) * (n ? n : 1));
    if (!v || !ix || !D->name) { free(v); free(ix); return ORC_E_OOM; }
    memcpy(v, a, sizeof(uint32_t) * na);
    memcpy(v + na, b, sizeof(uint32_t) * nb);
    for (int64_t i = 0; i < n; ++i) ix[i] = i;
    ukey_t u = { v };
    int st = stable_sort_idx(ix, n, cmp_u32key, &u);
    D->n = 0;
    for (int64_t i = 0; !st && i < n; ++i)
        if (D->n == 0 || D->name[D->n - 1] != v[ix[i]]) D->name[D->n++] = v[ix[i]];
    free(v); free(ix);
    return st;
}
static int64_t dict_find(const dict_t *D, uint32_t x) {
    int64_t a = 0, b = D->n;
    while (a < b) { int64_t m = a + (b - a) / 2; if (D->name[m] < x) a = m + 1; else b = m; }
    return (a < D->n && D->name[a] == x) ? a : -1;
}

/* summary: [0] kernels, [1] replayed, [2] direct, [3] broadcast, [4] unmatched
 *          [5] names with count mismatch, [6] replayed kernels left unmatched by
 *          the count rule, [7] dedup mismatches */
#define SUMMARY_N 8

static int check_dedup(int64_t K, const int32_t *layer, int32_t n_layers, const int32_t *class_of_layer,
                       int32_t n_classes, const int32_t *rep_of_class) {
    if (n_layers < 0 || n_classes < 0) return ORC_E_INVALID_ARG;
    for (int32_t l = 0; l < n_layers; ++l)
        if (class_of_layer[l] < 0 || class_of_layer[l] >= n_classes) return ORC_E_INVALID_ARG;
    for (int32_t c = 0; c < n_classes; ++c)
        if (rep_of_class[c] < 0 || rep_of_class[c] >= n_layers || class_of_layer[rep_of_class[c]] != c)
            return ORC_E_INVALID_ARG;
    for (int64_t k = 0; k < K; ++k)
        if (layer[k] >= n_layers || layer[k] < -1) return ORC_E_INVALID_ARG;
    return ORC_OK;
}

/* Matching.  mode: 0 skip-name, 1 prefix (Algorithm 1 as printed), 2 error.
 * dedup_on: 1 when layer deduplication applies (k_layer and tables given).
 * k_name is the matching key (the kernel name, or the (name, stream) key
 * with per-stream rows); k_layer_name is the kernel name itself, which the
 * broadcast of Sec. 3.7 compares between a layer and its class's
 * representative -- the two may run on different streams.
 * brute: 1 computes ordinals by rescanning all earlier records (definition
 * written out, O(K^2 + M^2)); 0 runs Algorithm 1's single pass with per-name
 * counters. */
int orc_match(int brute, int64_t K, const uint8_t *k_stream, const int64_t *k_start, const uint32_t *k_name,
              const uint32_t *k_layer_name, const int32_t *k_layer, int64_t M, const uint32_t *ncu_name,
              int dedup_on, int32_t n_layers,
              const int32_t *class_of_layer, int32_t n_classes, const int32_t *rep_of_class, int mode,
              int32_t *out_idx, uint8_t *out_kind, int64_t *summary) {
    if (mode < 0 || mode > 2) return ORC_E_INVALID_ARG;
    memset(summary, 0, sizeof(int64_t) * SUMMARY_N);
    summary[0] = K;
    dedup_on = dedup_on && k_layer != NULL;
    if (dedup_on) {
        int st = check_dedup(K, k_layer, n_layers, class_of_layer, n_classes, rep_of_class);
        if (st) return st;
    }
    int st = ORC_OK;
    int64_t *order = (int64_t *)malloc(sizeof(int64_t) * (K ? K : 1));
    uint8_t *replayed = (uint8_t *)malloc(K ? K : 1);
    int64_t *ord_k = (int64_t *)malloc(sizeof(int64_t) * (K ? K : 1));   /* ordinal o(k) */
    int64_t *ord_j = (int64_t *)malloc(sizeof(int64_t) * (M ? M : 1));   /* ordinal q(j) */
    dict_t D = { NULL, 0 };
    int64_t *cnt_k = NULL, *cnt_j = NULL, **rows = NULL;
    if (!order || !replayed || !ord_k || !ord_j) { st = ORC_E_OOM; goto done; }
    for (int64_t k = 0; k < K; ++k) order[k] = k;
    korder_t ko = { k_start, k_stream };
    if ((st = stable_sort_idx(order, K, cmp_time, &ko))) goto done;
    for (int64_t k = 0; k < K; ++k) {
        int32_t l = dedup_on ? k_layer[k] : -1;
        replayed[k] = (l < 0) || (rep_of_class[class_of_layer[l]] == l);
        summary[1] += replayed[k];
        out_idx[k] = -1;
        out_kind[k] = 0;
    }
    if ((st = dict_build(&D, k_name, K, ncu_name, M))) goto done;
    cnt_k = (int64_t *)calloc(D.n ? D.n : 1, sizeof(int64_t));
    cnt_j = (int64_t *)calloc(D.n ? D.n : 1, sizeof(int64_t));
    rows = (int64_t **)calloc(D.n ? D.n : 1, sizeof(int64_t *));
    if (!cnt_k || !cnt_j || !rows) { st = ORC_E_OOM; goto done; }

    /* ordinals */
    if (brute) {
        for (int64_t a = 0; a < K; ++a) {
            int64_t k = order[a], o = 0;
            if (!replayed[k]) continue;
            for (int64_t b = 0; b < a; ++b) o += replayed[order[b]] && k_name[order[b]] == k_name[k];
            ord_k[k] = o;
        }
        for (int64_t j = 0; j < M; ++j) {
            int64_t q = 0;
            for (int64_t i = 0; i < j; ++i) q += ncu_name[i] == ncu_name[j];
            ord_j[j] = q;
        }
    } else {
        for (int64_t a = 0; a < K; ++a) {              /* Algorithm 1: counter[name] */
            int64_t k = order[a];
            if (replayed[k]) ord_k[k] = cnt_k[dict_find(&D, k_name[k])]++;
        }
        for (int64_t j = 0; j < M; ++j) ord_j[j] = cnt_j[dict_find(&D, ncu_name[j])]++;
    }
    /* per-name totals (recounted plainly, both modes) and ncu rows by name */
    memset(cnt_k, 0, sizeof(int64_t) * D.n);
    memset(cnt_j, 0, sizeof(int64_t) * D.n);
    for (int64_t k = 0; k < K; ++k) if (replayed[k]) cnt_k[dict_find(&D, k_name[k])]++;
    for (int64_t j = 0; j < M; ++j) cnt_j[dict_find(&D, ncu_name[j])]++;
    for (int64_t n = 0; n < D.n; ++n) {
        rows[n] = (int64_t *)malloc(sizeof(int64_t) * (cnt_j[n] ? cnt_j[n] : 1));
        if (!rows[n]) { st = ORC_E_OOM; goto done; }
    }
    for (int64_t j = 0; j < M; ++j) rows[dict_find(&D, ncu_name[j])][ord_j[j]] = j;
    for (int64_t n = 0; n < D.n; ++n) if (cnt_k[n] != cnt_j[n]) summary[5]++;
    if (mode == MODE_ERROR && summary[5] > 0) { st = ORC_E_COUNT_MISMATCH; goto done; }

    /* direct assignment of replayed kernels */
    for (int64_t k = 0; k < K; ++k) {
        if (!replayed[k]) continue;
        int64_t n = dict_find(&D, k_name[k]);
        int ok = mode == MODE_SKIP_NAME ? (cnt_k[n] == cnt_j[n]) : (ord_k[k] < cnt_j[n]);
        if (ok) { out_idx[k] = (int32_t)rows[n][ord_k[k]]; out_kind[k] = 1; summary[2]++; }
        else summary[6]++;
    }

    /* broadcast to deduplicated layers (Sec. 3.7): position within the layer */
    if (dedup_on) {
        int64_t *pos = (int64_t *)malloc(sizeof(int64_t) * (K ? K : 1));
        int64_t *lay_cnt = (int64_t *)calloc(n_layers ? n_layers : 1, sizeof(int64_t));
        int64_t **lay_kern = (int64_t **)calloc(n_layers ? n_layers : 1, sizeof(int64_t *));
        if (!pos || !lay_cnt || !lay_kern) { free(pos); free(lay_cnt); free(lay_kern); st = ORC_E_OOM; goto done; }
        if (brute) {
            for (int64_t a = 0; a < K; ++a) {
                int64_t k = order[a], p = 0;
                if (k_layer[k] < 0) continue;
                for (int64_t b = 0; b < a; ++b) p += k_layer[order[b]] == k_layer[k];
                pos[k] = p;
            }
        } else {
            for (int64_t a = 0; a < K; ++a) {
                int64_t k = order[a];
                if (k_layer[k] >= 0) pos[k] = lay_cnt[k_layer[k]]++;
            }
            memset(lay_cnt, 0, sizeof(int64_t) * (n_layers ? n_layers : 1));
        }
        for (int64_t k = 0; k < K; ++k) if (k_layer[k] >= 0) lay_cnt[k_layer[k]]++;
        for (int32_t l = 0; l < n_layers; ++l) {
            lay_kern[l] = (int64_t *)malloc(sizeof(int64_t) * (lay_cnt[l] ? lay_cnt[l] : 1));
            if (!lay_kern[l]) st = ORC_E_OOM;
        }
        if (!st) {
            for (int64_t k = 0; k < K; ++k) if (k_layer[k] >= 0) lay_kern[k_layer[k]][pos[k]] = k;
            for (int64_t k = 0; k < K; ++k) {
                if (replayed[k]) continue;
                int32_t rep = rep_of_class[class_of_layer[k_layer[k]]];
                int64_t p = pos[k];
                int64_t src = p < lay_cnt[rep] ? lay_kern[rep][p] : -1;
                if (src >= 0 && k_layer_name[src] == k_layer_name[k] && out_idx[src] >= 0) {
                    out_idx[k] = out_idx[src]; out_kind[k] = 2; summary[3]++;
                } else {
                    summary[7]++;
                }
            }
        }
        for (int32_t l = 0; l < n_layers; ++l) free(lay_kern[l]);
        free(lay_kern); free(lay_cnt); free(pos);
        if (st) goto done;
    }
    for (int64_t k = 0; k < K; ++k) summary[4] += out_idx[k] < 0;
    if (mode == MODE_SKIP_NAME && summary[5] > 0) st = ORC_W_COUNT_MISMATCH;
    else if (mode == MODE_PREFIX && summary[6] > 0) st = ORC_W_COUNT_MISMATCH;
    else if (summary[7] > 0) st = ORC_W_DEDUP_MISMATCH;
done:
    if (rows) for (int64_t n = 0; n < D.n; ++n) free(rows[n]);
    free(rows); free(cnt_k); free(cnt_j); free(D.name);
    free(order); free(replayed); free(ord_k); free(ord_j);
    return st;
}

/* ------------------------------------------------------------------ aggregation */
typedef struct { double s, c; } nsum_t;      /* Neumaier running sum */
static void nadd(nsum_t *a, double x) {
    double t = a->s + x;
    if (fabs(a->s) >= fabs(x)) a->c += (a->s - t) + x; else a->c += (x - t) + a->s;
    a->s = t;
}
static double nval(const nsum_t *a) { return a->s + a->c; }

/* totals: [0] total_ns, [1] attributed_ns, [2] unattributed_ns, [3] kernels,
 *         [4] attributed kernels, [5] matched attributed kernels (int64);
 * fracs:  [0] attributed fraction, [1] unattributed fraction.
 * Outputs per op, SoA: kernel_count, total_duration_ns, matched_count (int64),
 * agg[c * n_ops + o] (fp64). */
int orc_aggregate(int64_t K, const int64_t *k_dur, const int32_t *range_of_kernel, int64_t R,
                  const uint32_t *r_op, int64_t M, const float *counters, const int32_t *ncu_idx,
                  int64_t n_ops, int64_t *kernel_count, int64_t *total_dur, int64_t *matched,
                  double *agg, int64_t *totals, double *fracs) {
    for (int64_t k = 0; k < K; ++k) {
        int32_t r = range_of_kernel[k], j = ncu_idx ? ncu_idx[k] : -1;
        if (k_dur[k] < 0 || r < -1 || r >= R || j < -1 || j >= M) return ORC_E_INVALID_ARG;
        if (r >= 0 && (int64_t)r_op[r] >= n_ops) return ORC_E_INVALID_ARG;
        if (r >= 0 && j >= 0)
            for (int c = 0; c < NC; ++c) if (isinf(counters[(int64_t)j * NC + c])) return ORC_E_INVALID_ARG;
    }
    nsum_t *num = (nsum_t *)calloc((size_t)(n_ops ? n_ops : 1) * NC, sizeof(nsum_t));
    int64_t *den = (int64_t *)calloc((size_t)(n_ops ? n_ops : 1) * NC, sizeof(int64_t));
    double *mx = (double *)malloc(sizeof(double) * (size_t)(n_ops ? n_ops : 1) * NC);
    int64_t *seen = (int64_t *)calloc((size_t)(n_ops ? n_ops : 1) * NC, sizeof(int64_t));
    if (!num || !den || !mx || !seen) { free(num); free(den); free(mx); free(seen); return ORC_E_OOM; }
    for (int64_t o = 0; o < n_ops; ++o) { kernel_count[o] = 0; total_dur[o] = 0; matched[o] = 0; }
    int64_t tot = 0, att = 0, natt = 0, nmatch = 0;
    for (int64_t k = 0; k < K; ++k) {
        int64_t d = k_dur[k];
        tot += d;
        int32_t r = range_of_kernel[k];
        if (r < 0) continue;
        int64_t o = r_op[r];
        att += d; natt++;
        kernel_count[o]++;
        total_dur[o] += d;
        int32_t j = ncu_idx ? ncu_idx[k] : -1;
        if (j < 0) continue;
        matched[o]++; nmatch++;
        for (int c = 0; c < NC; ++c) {
            double m = counters[(int64_t)j * NC + c];
            if (isnan(m)) continue;                      /* null counter */
            size_t at = (size_t)c * n_ops + o;
            if (AGG_RULE[c] == AGG_SUM) nadd(&num[at], m);
            else if (AGG_RULE[c] == AGG_DW) { nadd(&num[at], m * (double)d); den[at] += d; }
            else mx[at] = seen[at] ? (m > mx[at] ? m : mx[at]) : m;
            seen[at]++;
        }
    }
    for (int c = 0; c < NC; ++c) {
        for (int64_t o = 0; o < n_ops; ++o) {
            size_t at = (size_t)c * n_ops + o;
            double v = NAN;
            if (seen[at]) {
                if (AGG_RULE[c] == AGG_SUM) v = nval(&num[at]);
                else if (AGG_RULE[c] == AGG_MAX) v = mx[at];
                else if (den[at] > 0) v = nval(&num[at]) / (double)den[at];
            }
            agg[at] = v;
        }
    }
    totals[0] = tot; totals[1] = att; totals[2] = tot - att; totals[3] = K; totals[4] = natt; totals[5] = nmatch;
    fracs[0] = tot > 0 ? (double)att / (double)tot : NAN;
    fracs[1] = tot > 0 ? (double)(tot - att) / (double)tot : NAN;
    free(num); free(den); free(mx); free(seen);
    return ORC_OK;
}

/* ------------------------------------------------------------------ attribution tiers
 * Fig. 2, tried per kernel in this order:
 *   HIGH      the torch.profiler correlation map (Sec. 3.4) holds an entry for
 *             the kernel's (name, invocation index); the invocation index is
 *             the number of earlier kernels (time order) with the same name;
 *   NVTX      the kernel has an enclosing operator range (Algorithm 2's
 *             result, range_of_kernel >= 0);
 *   INDUCTOR  the Inductor fusion map (Sec. 3.6) names an operator for the
 *             kernel's name;
 *   otherwise the kernel is unattributed.
 * The fusion map enriches every tier: fused_with = the name's fusion
 * operator; is_fused = its operator list is longer than one, or (NVTX tier)
 * the walk collected more than one operator range.
 * A map entry that names a launch must be the only entry for that pair; map
 * entries naming no launch are ignored.
 * brute: invocation indices by rescanning every earlier kernel, map lookups
 * by scanning the whole map; otherwise per-name counters and a sorted map.
 * summary: [0] kernels [1] high [2] nvtx [3] inductor [4] none [5] fused
 *          [6] map entries that named a launch */
#define ATTR_SUMMARY_N 7
#define OP_NONE 0xFFFFFFFFu
enum { TIER_NONE = 0, TIER_HIGH = 1, TIER_NVTX = 2, TIER_INDUCTOR = 3 };

typedef struct { const uint32_t *name, *inv; } corrkey_t;
static int cmp_corr(int64_t a, int64_t b, const void *ctx) {
    const corrkey_t *c = (const corrkey_t *)ctx;
    if (c->name[a] != c->name[b]) return c->name[a] < c->name[b] ? -1 : 1;
    if (c->inv[a] != c->inv[b]) return c->inv[a] < c->inv[b] ? -1 : 1;
    return 0;
}

int orc_attribute(int brute, int64_t K, const uint8_t *k_stream, const int64_t *k_start, const uint32_t *k_name,
                  const int32_t *rok, const uint8_t *nop, int64_t R, const uint32_t *r_op, uint32_t n_ops,
                  int64_t NM, const uint32_t *c_name, const uint32_t *c_inv, const uint32_t *c_op, int64_t NF,
                  const uint32_t *f_op, const uint8_t *f_len, uint32_t *op_of_kernel, uint8_t *tier,
                  uint32_t *fused_with, uint8_t *is_fused, int64_t *summary) {
    memset(summary, 0, sizeof(int64_t) * ATTR_SUMMARY_N);
    summary[0] = K;
    for (int64_t k = 0; k < K; ++k) {
        if (rok[k] < -1 || rok[k] >= R) return ORC_E_INVALID_ARG;
        if (rok[k] >= 0 && r_op[rok[k]] >= n_ops) return ORC_E_INVALID_ARG;
    }
    for (int64_t e = 0; e < NM; ++e) if (c_op[e] >= n_ops) return ORC_E_INVALID_ARG;
    for (int64_t n = 0; n < NF; ++n) if (f_op[n] != OP_NONE && f_op[n] >= n_ops) return ORC_E_INVALID_ARG;

    int st = ORC_OK;
    int64_t *order = (int64_t *)malloc(sizeof(int64_t) * (K ? K : 1));
    uint32_t *inv = (uint32_t *)malloc(sizeof(uint32_t) * (K ? K : 1));
    int64_t *cix = (int64_t *)malloc(sizeof(int64_t) * (NM ? NM : 1));
    int64_t *cnt = NULL;
    dict_t D = { NULL, 0 };
    if (!order || !inv || !cix) { st = ORC_E_OOM; goto done; }
    for (int64_t k = 0; k < K; ++k) order[k] = k;
    korder_t ko = { k_start, k_stream };
    if ((st = stable_sort_idx(order, K, cmp_time, &ko))) goto done;

    /* invocation index of every kernel */
    if (brute) {
        for (int64_t a = 0; a < K; ++a) {
            uint32_t c = 0;
            for (int64_t b = 0; b < a; ++b) c += k_name[order[b]] == k_name[order[a]];
            inv[order[a]] = c;
        }
    } else {
        if ((st = dict_build(&D, k_name, K, k_name, 0))) goto done;
        cnt = (int64_t *)calloc(D.n ? D.n : 1, sizeof(int64_t));
        if (!cnt) { st = ORC_E_OOM; goto done; }
        for (int64_t a = 0; a < K; ++a) {
            int64_t k = order[a];
            inv[k] = (uint32_t)cnt[dict_find(&D, k_name[k])]++;
        }
    }
    /* the map, sorted by (name, invocation) unless scanned whole */
    for (int64_t e = 0; e < NM; ++e) cix[e] = e;
    corrkey_t ck = { c_name, c_inv };
    if (!brute && (st = stable_sort_idx(cix, NM, cmp_corr, &ck))) goto done;

    for (int64_t k = 0; k < K; ++k) {
        /* HIGH: entries for (name, invocation index) */
        int64_t hits = 0, hit = -1;
        if (brute) {
            for (int64_t e = 0; e < NM; ++e)
                if (c_name[e] == k_name[k] && c_inv[e] == inv[k]) { hits++; hit = e; }
        } else {
            int64_t lo = 0, hi = NM;          /* first entry >= (name, inv) */
            while (lo < hi) {
                int64_t m = lo + (hi - lo) / 2, e = cix[m];
                if (c_name[e] < k_name[k] || (c_name[e] == k_name[k] && c_inv[e] < inv[k])) lo = m + 1; else hi = m;
            }
            for (int64_t m = lo; m < NM && c_name[cix[m]] == k_name[k] && c_inv[cix[m]] == inv[k]; ++m) {
                hits++;
                hit = cix[m];
            }
        }
        if (hits > 1) { st = ORC_E_INVALID_ARG; goto done; }
        summary[6] += hits;
        const uint32_t fo = (int64_t)k_name[k] < NF ? f_op[k_name[k]] : OP_NONE;
        const unsigned fl = ((int64_t)k_name[k] < NF && f_len) ? f_len[k_name[k]] : 1u;
        uint32_t op = OP_NONE;
        uint8_t t = TIER_NONE;
        if (hits == 1) { op = c_op[hit]; t = TIER_HIGH; }
        else if (rok[k] >= 0) { op = r_op[rok[k]]; t = TIER_NVTX; }
        else if (fo != OP_NONE) { op = fo; t = TIER_INDUCTOR; }
        const int fused = (fo != OP_NONE && fl > 1) || (t == TIER_NVTX && nop && nop[k] > 1);
        op_of_kernel[k] = op;
        tier[k] = t;
        fused_with[k] = fo;
        is_fused[k] = (uint8_t)fused;
        summary[1] += t == TIER_HIGH;
        summary[2] += t == TIER_NVTX;
        summary[3] += t == TIER_INDUCTOR;
        summary[4] += t == TIER_NONE;
        summary[5] += fused;
    }
done:
    free(order); free(inv); free(cix); free(cnt); free(D.name);
    return st;
}
