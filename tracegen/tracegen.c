/*
 * tracegen.c -- seeded synthetic traces shaped like an Nsight Systems export
 * (kernel records + NVTX ranges per stream) and an Nsight Compute export
 * (per-launch counter rows in launch order).
 *
 * This module only draws inputs.  It holds none of the attribution arithmetic:
 * it never decides which range encloses which kernel, never matches ncu rows,
 * never aggregates.  Both the CPU oracle and the CUDA library consume what it
 * writes.
 *
 * Random numbers: SplitMix64 (Steele, Lea & Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014).  Every array draws from its
 * own key, so streams can be simulated in parallel and counters are
 * counter-based (value = f(key, row, column)).
 *
 * Ranges are produced by a push/pop simulation per stream, so every stream's
 * range family is laminar by construction: a range pushed while another is
 * open is popped first.  A range's depth is the number of ranges open when it
 * was pushed.  Structural ranges (steps, layers, blocks) carry op id
 * TG_STRUCTURAL, namespaced non-op ranges carry TG_NONOP, every other range
 * is an operator dispatch and gets its own op id, numbered in global start
 * order.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define TG_STRUCTURAL 0xFFFFFFFFu
#define TG_NONOP 0xFFFFFFFEu
#define TG_MAX_DEPTH 32
#define TG_NCOUNTERS 20

typedef struct {
    uint64_t seed;
    int32_t shape;            /* 0 = random operator trees, 1 = layered templates */
    int32_t n_streams;
    int64_t n_kernels;        /* shape 0: total kernels (split evenly over streams) */
    int32_t max_depth;        /* depth values are 0 .. max_depth-1 */
    int32_t n_names;
    double zipf_s;
    double dur_median_ns, dur_sigma;
    double gap_mean_ns;
    double delta_mean_ns;     /* host time between a push and the next event */
    double p_zero_delta;      /* probability that such a delta is exactly 0 */
    double uncovered_frac;    /* target share of kernels outside every range */
    int32_t uncovered_by_time;/* 1: share measured over durations */
    double bb_run_mean;       /* mean length of a run of uncovered kernels */
    /* shape 0 */
    double kids_mean;         /* mean children of a range node, beyond the first */
    double p_kernel_child;    /* probability a child is a kernel, not a sub-range */
    double p_nonop;           /* share of sub-ranges that are namespaced non-ops */
    double p_struct_inner;    /* share of sub-ranges that are structural */
    double p_empty;           /* operator ranges that launch nothing */
    double p_chain;           /* a range whose only child is one sub-range */
    /* shape 1 */
    int32_t n_iters, n_slots, n_classes;
    int32_t tmpl_len[8];      /* kernels per layer template, per class */
    int32_t layer_per_stream; /* 1: layer id = stream * n_slots + slot */
    int32_t step_kernels;     /* kernels launched directly inside each step */
    int32_t dedup;            /* ncu rows only for representative layers */
    /* counters */
    int32_t counter_dist;     /* 0 uniform [lo,hi], 1 log-uniform [lo,hi] */
    double counter_lo, counter_hi;
    double nan_frac;          /* share of counter cells that are null (NaN) */
    uint32_t nan_mask;        /* counter columns that are null in every row */
    int32_t shuffle;          /* permute kernel and range arrays after merging */
} tg_config;

/* ---------------------------------------------------------------- RNG */
static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}
#define GOLDEN 0x9e3779b97f4a7c15ULL
typedef struct { uint64_t s; } rng_t;
static inline uint64_t rng_next(rng_t *r) { r->s += GOLDEN; return mix64(r->s); }
static inline double rng_u01(rng_t *r) { return (double)(rng_next(r) >> 11) * 0x1.0p-53; }
static inline double rng_u01_open(rng_t *r) { return ((double)(rng_next(r) >> 11) + 0.5) * 0x1.0p-53; }
static rng_t rng_key(uint64_t seed, uint64_t a, uint64_t b) {
    rng_t r; r.s = mix64(seed ^ mix64(a * 0x632be59bd9b4e019ULL + 1) ^ mix64(b + 0x8cb92ba72f3d8dd7ULL));
    return r;
}
static inline double rng_normal(rng_t *r) {   /* Box-Muller, one of the pair */
    double u1 = rng_u01_open(r), u2 = rng_u01(r);
    return sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
}
static inline double rng_exp(rng_t *r, double mean) { return -mean * log(rng_u01_open(r)); }
static inline int rng_geom(rng_t *r, double mean) {   /* >= 0, given mean */
    if (mean <= 0) return 0;
    double p = 1.0 / (1.0 + mean);
    int n = (int)floor(log(rng_u01_open(r)) / log(1.0 - p));
    return n < 0 ? 0 : (n > 1000 ? 1000 : n);
}

/* ---------------------------------------------------------------- growable arrays */
typedef struct { int64_t t, dur; uint32_t name; int32_t layer; } kern_t;
typedef struct { int64_t start, end; uint32_t kind; uint8_t depth; } range_t;
typedef struct { kern_t *k; int64_t nk, ck; range_t *r; int64_t nr, cr; } strm_t;

static void push_k(strm_t *s, kern_t v) {
    if (s->nk == s->ck) { s->ck = s->ck ? s->ck * 2 : 1024; s->k = (kern_t *)realloc(s->k, s->ck * sizeof(kern_t)); }
    s->k[s->nk++] = v;
}
static int64_t push_r(strm_t *s, range_t v) {
    if (s->nr == s->cr) { s->cr = s->cr ? s->cr * 2 : 1024; s->r = (range_t *)realloc(s->r, s->cr * sizeof(range_t)); }
    s->r[s->nr] = v; return s->nr++;
}

/* ---------------------------------------------------------------- per-stream simulation */
typedef struct {
    const tg_config *c;
    const double *zipf_cdf;
    strm_t *s;
    rng_t rng;
    int64_t t;                 /* host clock of this stream, ns */
    int64_t quota, emitted;    /* kernels this stream may emit / has emitted */
    double cov_w, unc_w;       /* covered / uncovered weight so far */
    int64_t open[TG_MAX_DEPTH];
    int depth;
    int32_t layer;             /* layer tag of kernels emitted now, -1 outside */
} sim_t;

static uint32_t draw_name(sim_t *m) {
    double u = rng_u01(&m->rng);
    int lo = 0, hi = m->c->n_names - 1;
    while (lo < hi) { int mid = (lo + hi) / 2; if (m->zipf_cdf[mid] > u) hi = mid; else lo = mid + 1; }
    return (uint32_t)lo;
}
static int64_t draw_delta(sim_t *m) {
    if (rng_u01(&m->rng) < m->c->p_zero_delta) return 0;
    return (int64_t)llround(rng_exp(&m->rng, m->c->delta_mean_ns));
}
static void emit_kernel(sim_t *m, uint32_t name, int covered) {
    if (m->emitted >= m->quota) return;
    double z = rng_normal(&m->rng);
    double d = floor(m->c->dur_median_ns * exp(m->c->dur_sigma * z) + 0.5);
    if (d < 0) d = 0;
    if (d > 1e12) d = 1e12;
    int64_t dur = (int64_t)d;
    int64_t gap = (int64_t)llround(rng_exp(&m->rng, m->c->gap_mean_ns));
    kern_t k = { m->t, dur, name, m->layer };
    push_k(m->s, k);
    m->emitted++;
    double w = m->c->uncovered_by_time ? (double)dur : 1.0;
    if (covered) m->cov_w += w; else m->unc_w += w;
    m->t += dur + gap;
}
static void push_range(sim_t *m, uint32_t kind) {
    range_t r = { m->t, -1, kind, (uint8_t)m->depth };
    m->open[m->depth++] = push_r(m->s, r);
    m->t += draw_delta(m);
}
static void pop_range(sim_t *m) {
    int64_t id = m->open[--m->depth];
    m->s->r[id].end = m->t;
    m->t += draw_delta(m);
}

/* shape 0: one random operator tree below an open range at depth m->depth */
static void gen_node(sim_t *m, uint32_t kind) {
    const tg_config *c = m->c;
    push_range(m, kind);
    int d = m->depth;          /* depth a child range would get */
    if (kind < TG_NONOP && rng_u01(&m->rng) < c->p_empty) {
        /* an operator that launches nothing (a view, a metadata op) */
    } else if (d < c->max_depth && rng_u01(&m->rng) < c->p_chain) {
        uint32_t ck = rng_u01(&m->rng) < c->p_nonop ? TG_NONOP : 0;
        gen_node(m, ck);
    } else {
        int n = 1 + rng_geom(&m->rng, c->kids_mean);
        for (int i = 0; i < n; ++i) {
            if (d < c->max_depth && rng_u01(&m->rng) >= c->p_kernel_child) {
                double u = rng_u01(&m->rng);
                uint32_t ck = u < c->p_struct_inner ? TG_STRUCTURAL
                            : (u < c->p_struct_inner + c->p_nonop ? TG_NONOP : 0);
                gen_node(m, ck);
            } else {
                emit_kernel(m, draw_name(m), 1);
            }
        }
    }
    pop_range(m);
}

static int uncovered_due(sim_t *m) {
    double tot = m->cov_w + m->unc_w;
    return m->unc_w < m->c->uncovered_frac * tot || (tot == 0 && m->c->uncovered_frac >= 1.0);
}

static void sim_random(sim_t *m) {
    const tg_config *c = m->c;
    while (m->emitted < m->quota) {
        if (c->uncovered_frac > 0 && uncovered_due(m)) {
            int n = 1 + rng_geom(&m->rng, c->bb_run_mean - 1.0);
            for (int i = 0; i < n; ++i) emit_kernel(m, draw_name(m), 0);
            m->t += draw_delta(m);
        } else if (c->max_depth <= 1) {
            gen_node(m, 0);
        } else {
            /* a structural step at depth 0 holding operator trees */
            push_range(m, TG_STRUCTURAL);
            int n = 1 + rng_geom(&m->rng, c->kids_mean + 1.0);
            for (int i = 0; i < n && m->emitted < m->quota; ++i) {
                double u = rng_u01(&m->rng);
                gen_node(m, u < c->p_nonop ? TG_NONOP : 0);
            }
            pop_range(m);
        }
    }
}

/* shape 1: layer templates.  A template is a fixed event list replayed for
 * every instance of a class; only durations and gaps are redrawn. */
enum { EV_PUSH_STRUCT = 1, EV_PUSH_OP, EV_PUSH_NONOP, EV_POP, EV_KERNEL };
typedef struct { int kind; uint32_t name; } tev_t;
typedef struct { tev_t *ev; int n, cap; } tmpl_t;
static void tadd(tmpl_t *t, int kind, uint32_t name) {
    if (t->n == t->cap) { t->cap = t->cap ? t->cap * 2 : 64; t->ev = (tev_t *)realloc(t->ev, t->cap * sizeof(tev_t)); }
    t->ev[t->n].kind = kind; t->ev[t->n].name = name; t->n++;
}
static void build_template(tmpl_t *t, const tg_config *c, const double *cdf, int cls) {
    sim_t m; memset(&m, 0, sizeof m); m.c = c; m.zipf_cdf = cdf;
    m.rng = rng_key(c->seed, 0x7e3a11, (uint64_t)cls);
    int left = c->tmpl_len[cls];
    /* layer (depth 1) > 2 blocks (depth 2) > operators (3) > sub-operators (4) > wrapped (5) */
    int in_block[2] = { left / 2, left - left / 2 };
    for (int b = 0; b < 2; ++b) {
        tadd(t, EV_PUSH_STRUCT, 0);
        int k = in_block[b];
        while (k > 0) {
            double u = rng_u01(&m.rng);
            if (u < 0.12) {                    /* a kernel directly inside a block */
                tadd(t, EV_KERNEL, draw_name(&m)); k--;
            } else if (u < 0.15) {             /* an operator that launches nothing */
                tadd(t, EV_PUSH_OP, 0); tadd(t, EV_POP, 0);
            } else if (u < 0.25 && k >= 3) {   /* an operator with a nested operator */
                tadd(t, EV_PUSH_OP, 0);
                tadd(t, EV_KERNEL, draw_name(&m)); k--;
                tadd(t, EV_PUSH_OP, 0);
                int n = 1 + (int)(rng_u01(&m.rng) * 3); if (n > k) n = k;
                for (int i = 0; i < n; ++i) { tadd(t, EV_KERNEL, draw_name(&m)); k--; }
                tadd(t, EV_POP, 0);
                tadd(t, EV_POP, 0);
            } else if (u < 0.30 && k >= 2) {   /* operator > non-op wrapper > operator */
                tadd(t, EV_PUSH_OP, 0);
                tadd(t, EV_PUSH_NONOP, 0);
                tadd(t, EV_PUSH_OP, 0);
                int n = 1 + (int)(rng_u01(&m.rng) * 2); if (n > k) n = k;
                for (int i = 0; i < n; ++i) { tadd(t, EV_KERNEL, draw_name(&m)); k--; }
                tadd(t, EV_POP, 0);
                tadd(t, EV_POP, 0);
                tadd(t, EV_POP, 0);
            } else {                           /* a plain operator with 1..13 kernels */
                tadd(t, EV_PUSH_OP, 0);
                int n = 1 + (int)(rng_u01(&m.rng) * 13); if (n > k) n = k;
                for (int i = 0; i < n; ++i) { tadd(t, EV_KERNEL, draw_name(&m)); k--; }
                tadd(t, EV_POP, 0);
            }
        }
        tadd(t, EV_POP, 0);
    }
}

static void sim_layered(sim_t *m, int stream, tmpl_t *tm) {
    const tg_config *c = m->c;
    m->quota = INT64_MAX;
    for (int it = 0; it < c->n_iters; ++it) {
        m->layer = -1;
        push_range(m, TG_STRUCTURAL);                      /* the profiler step */
        for (int i = 0; i < c->step_kernels; ++i) emit_kernel(m, draw_name(m), 1);
        for (int slot = 0; slot < c->n_slots; ++slot) {
            int cls = slot % c->n_classes;
            m->layer = c->layer_per_stream ? stream * c->n_slots + slot : slot;
            push_range(m, TG_STRUCTURAL);                  /* the layer */
            const tmpl_t *t = &tm[cls];
            for (int e = 0; e < t->n; ++e) {
                switch (t->ev[e].kind) {
                case EV_PUSH_STRUCT: push_range(m, TG_STRUCTURAL); break;
                case EV_PUSH_OP: push_range(m, 0); break;
                case EV_PUSH_NONOP: push_range(m, TG_NONOP); break;
                case EV_POP: pop_range(m); break;
                default: emit_kernel(m, t->ev[e].name, 1); break;
                }
            }
            pop_range(m);
            m->layer = -1;
        }
        pop_range(m);
        m->t += draw_delta(m);
        if (c->uncovered_frac > 0 && uncovered_due(m)) {  /* e.g. an optimizer step outside ranges */
            int n = 1 + rng_geom(&m->rng, c->bb_run_mean - 1.0);
            for (int i = 0; i < n; ++i) emit_kernel(m, draw_name(m), 0);
        }
    }
}

/* ---------------------------------------------------------------- k-way merge */
typedef struct { int64_t key; int32_t stream; int64_t pos; } hnode_t;
static int hless(const hnode_t *a, const hnode_t *b) {
    return a->key < b->key || (a->key == b->key && a->stream < b->stream);
}
static void hsift(hnode_t *h, int n, int i) {
    for (;;) {
        int l = 2 * i + 1, r = l + 1, s = i;
        if (l < n && hless(&h[l], &h[s])) s = l;
        if (r < n && hless(&h[r], &h[s])) s = r;
        if (s == i) return;
        hnode_t x = h[i]; h[i] = h[s]; h[s] = x; i = s;
    }
}

/* ---------------------------------------------------------------- result handle */
typedef struct {
    int64_t K, R, M, n_ops;
    int32_t n_layers, n_classes, has_layer;
    uint8_t *k_stream; int64_t *k_start, *k_dur; uint32_t *k_name; int32_t *k_layer;
    uint8_t *r_stream; int64_t *r_start, *r_end; uint8_t *r_depth; uint32_t *r_op;
    uint32_t *ncu_name;
    int32_t *class_of_layer, *rep_of_class;
    tg_config cfg;
} tg_trace;

static void shuffle_perm(int64_t *p, int64_t n, rng_t *r) {
    for (int64_t i = 0; i < n; ++i) p[i] = i;
    for (int64_t i = n - 1; i > 0; --i) {
        int64_t j = (int64_t)(rng_next(r) % (uint64_t)(i + 1));
        int64_t x = p[i]; p[i] = p[j]; p[j] = x;
    }
}

int tg_generate(const tg_config *cfg, tg_trace **out) {
    *out = NULL;
    if (cfg->n_streams < 1 || cfg->n_streams > 256 || cfg->max_depth < 1 || cfg->max_depth > TG_MAX_DEPTH ||
        cfg->n_names < 1 || cfg->n_classes > 8) return -1;
    int S = cfg->n_streams;
    double *cdf = (double *)malloc(sizeof(double) * cfg->n_names);
    double acc = 0;
    for (int i = 0; i < cfg->n_names; ++i) { acc += pow((double)(i + 1), -cfg->zipf_s); cdf[i] = acc; }
    for (int i = 0; i < cfg->n_names; ++i) cdf[i] /= acc;
    cdf[cfg->n_names - 1] = 2.0;

    tmpl_t tm[8]; memset(tm, 0, sizeof tm);
    if (cfg->shape == 1)
        for (int c = 0; c < cfg->n_classes; ++c) build_template(&tm[c], cfg, cdf, c);

    strm_t *st = (strm_t *)calloc(S, sizeof(strm_t));
#pragma omp parallel for schedule(dynamic, 1)
    for (int s = 0; s < S; ++s) {
        sim_t m; memset(&m, 0, sizeof m);
        m.c = cfg; m.zipf_cdf = cdf; m.s = &st[s]; m.layer = -1;
        m.rng = rng_key(cfg->seed, 0x5eed, (uint64_t)s);
        m.t = (int64_t)(rng_u01(&m.rng) * cfg->gap_mean_ns * 4.0);
        if (cfg->shape == 1) {
            sim_layered(&m, s, tm);
        } else {
            m.quota = cfg->n_kernels / S + (s < cfg->n_kernels % S ? 1 : 0);
            sim_random(&m);
        }
    }
    for (int c = 0; c < 8; ++c) free(tm[c].ev);
    free(cdf);

    tg_trace *tr = (tg_trace *)calloc(1, sizeof(tg_trace));
    tr->cfg = *cfg;
    int64_t K = 0, R = 0;
    for (int s = 0; s < S; ++s) { K += st[s].nk; R += st[s].nr; }
    tr->K = K; tr->R = R;
    tr->has_layer = cfg->shape == 1;
    tr->k_stream = (uint8_t *)malloc(K ? K : 1);
    tr->k_start = (int64_t *)malloc(8 * (K ? K : 1));
    tr->k_dur = (int64_t *)malloc(8 * (K ? K : 1));
    tr->k_name = (uint32_t *)malloc(4 * (K ? K : 1));
    tr->k_layer = (int32_t *)malloc(4 * (K ? K : 1));
    tr->r_stream = (uint8_t *)malloc(R ? R : 1);
    tr->r_start = (int64_t *)malloc(8 * (R ? R : 1));
    tr->r_end = (int64_t *)malloc(8 * (R ? R : 1));
    tr->r_depth = (uint8_t *)malloc(R ? R : 1);
    tr->r_op = (uint32_t *)malloc(4 * (R ? R : 1));

    /* merge kernels by (start, stream); per-stream order is already by start */
    hnode_t *h = (hnode_t *)malloc(sizeof(hnode_t) * S);
    int hn = 0;
    for (int s = 0; s < S; ++s) if (st[s].nk) { h[hn].key = st[s].k[0].t; h[hn].stream = s; h[hn].pos = 0; hn++; }
    for (int i = hn / 2 - 1; i >= 0; --i) hsift(h, hn, i);
    for (int64_t o = 0; hn > 0; ++o) {
        strm_t *q = &st[h[0].stream]; const kern_t *k = &q->k[h[0].pos];
        tr->k_stream[o] = (uint8_t)h[0].stream; tr->k_start[o] = k->t; tr->k_dur[o] = k->dur;
        tr->k_name[o] = k->name; tr->k_layer[o] = k->layer;
        if (++h[0].pos < q->nk) h[0].key = q->k[h[0].pos].t; else h[0] = h[--hn];
        hsift(h, hn, 0);
    }
    /* merge ranges by (start, stream); per-stream order is push order */
    hn = 0;
    for (int s = 0; s < S; ++s) if (st[s].nr) { h[hn].key = st[s].r[0].start; h[hn].stream = s; h[hn].pos = 0; hn++; }
    for (int i = hn / 2 - 1; i >= 0; --i) hsift(h, hn, i);
    uint32_t next_op = 0;
    for (int64_t o = 0; hn > 0; ++o) {
        strm_t *q = &st[h[0].stream]; const range_t *r = &q->r[h[0].pos];
        tr->r_stream[o] = (uint8_t)h[0].stream; tr->r_start[o] = r->start; tr->r_end[o] = r->end;
        tr->r_depth[o] = r->depth;
        tr->r_op[o] = r->kind ? r->kind : next_op++;
        if (++h[0].pos < q->nr) h[0].key = q->r[h[0].pos].start; else h[0] = h[--hn];
        hsift(h, hn, 0);
    }
    free(h);
    for (int s = 0; s < S; ++s) { free(st[s].k); free(st[s].r); }
    free(st);
    tr->n_ops = next_op;

    /* layers, classes, representatives */
    if (cfg->shape == 1) {
        tr->n_layers = cfg->layer_per_stream ? S * cfg->n_slots : cfg->n_slots;
        tr->n_classes = cfg->n_classes;
        tr->class_of_layer = (int32_t *)malloc(4 * tr->n_layers);
        tr->rep_of_class = (int32_t *)malloc(4 * tr->n_classes);
        for (int c = 0; c < tr->n_classes; ++c) tr->rep_of_class[c] = -1;
        for (int l = 0; l < tr->n_layers; ++l) {
            int c = (l % cfg->n_slots) % cfg->n_classes;
            tr->class_of_layer[l] = c;
            if (tr->rep_of_class[c] < 0) tr->rep_of_class[c] = l;
        }
    }

    /* ncu rows: one per replayed launch, in launch (= time) order */
    int64_t M = 0;
    tr->ncu_name = (uint32_t *)malloc(4 * (K ? K : 1));
    for (int64_t i = 0; i < K; ++i) {
        int32_t l = tr->k_layer[i];
        int replayed = !(cfg->shape == 1 && cfg->dedup) || l < 0 || tr->rep_of_class[tr->class_of_layer[l]] == l;
        if (replayed) tr->ncu_name[M++] = tr->k_name[i];
    }
    tr->M = M;

    if (cfg->shuffle) {
        rng_t r = rng_key(cfg->seed, 0x5f1e, 1);
        int64_t n = K > R ? K : R;
        int64_t *p = (int64_t *)malloc(8 * (n ? n : 1));
        shuffle_perm(p, K, &r);
        uint8_t *a8 = (uint8_t *)malloc(K ? K : 1); int64_t *a64 = (int64_t *)malloc(8 * (K ? K : 1));
        uint32_t *a32 = (uint32_t *)malloc(4 * (K ? K : 1));
#define PERMUTE(arr, tmp, n_) do { for (int64_t i = 0; i < (n_); ++i) tmp[i] = arr[p[i]]; memcpy(arr, tmp, sizeof(*arr) * (n_)); } while (0)
        PERMUTE(tr->k_stream, a8, K); PERMUTE(tr->k_start, a64, K); PERMUTE(tr->k_dur, a64, K);
        PERMUTE(tr->k_name, a32, K); PERMUTE(tr->k_layer, ((int32_t *)a32), K);
        shuffle_perm(p, R, &r);
        uint8_t *b8 = (uint8_t *)malloc(R ? R : 1); int64_t *b64 = (int64_t *)malloc(8 * (R ? R : 1));
        uint32_t *b32 = (uint32_t *)malloc(4 * (R ? R : 1));
        PERMUTE(tr->r_stream, b8, R); PERMUTE(tr->r_start, b64, R); PERMUTE(tr->r_end, b64, R);
        PERMUTE(tr->r_depth, b8, R); PERMUTE(tr->r_op, b32, R);
#undef PERMUTE
        free(a8); free(a64); free(a32); free(b8); free(b64); free(b32); free(p);
    }
    *out = tr;
    return 0;
}

void tg_sizes(const tg_trace *t, int64_t *out) {
    out[0] = t->K; out[1] = t->R; out[2] = t->M; out[3] = t->n_ops;
    out[4] = t->n_layers; out[5] = t->n_classes; out[6] = t->has_layer;
}

/* Copy into caller buffers (NULL = skip).  Counters are drawn here, straight
 * into the caller's n x 20 row-major float buffer. */
void tg_copy(const tg_trace *t, uint8_t *k_stream, int64_t *k_start, int64_t *k_dur, uint32_t *k_name,
             int32_t *k_layer, uint8_t *r_stream, int64_t *r_start, int64_t *r_end, uint8_t *r_depth,
             uint32_t *r_op, uint32_t *ncu_name, float *counters, int32_t *class_of_layer,
             int32_t *rep_of_class) {
    int64_t K = t->K, R = t->R, M = t->M;
    if (k_stream) memcpy(k_stream, t->k_stream, K);
    if (k_start) memcpy(k_start, t->k_start, 8 * K);
    if (k_dur) memcpy(k_dur, t->k_dur, 8 * K);
    if (k_name) memcpy(k_name, t->k_name, 4 * K);
    if (k_layer && t->has_layer) memcpy(k_layer, t->k_layer, 4 * K);
    if (r_stream) memcpy(r_stream, t->r_stream, R);
    if (r_start) memcpy(r_start, t->r_start, 8 * R);
    if (r_end) memcpy(r_end, t->r_end, 8 * R);
    if (r_depth) memcpy(r_depth, t->r_depth, R);
    if (r_op) memcpy(r_op, t->r_op, 4 * R);
    if (ncu_name) memcpy(ncu_name, t->ncu_name, 4 * M);
    if (class_of_layer && t->n_layers) memcpy(class_of_layer, t->class_of_layer, 4 * t->n_layers);
    if (rep_of_class && t->n_classes) memcpy(rep_of_class, t->rep_of_class, 4 * t->n_classes);
    if (counters) {
        const tg_config *c = &t->cfg;
        uint64_t key = mix64(c->seed ^ 0xc0ffee123ULL);
        double lo = c->counter_lo, hi = c->counter_hi;
        double llo = c->counter_dist == 1 ? log(lo) : 0, lhi = c->counter_dist == 1 ? log(hi) : 0;
#pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < M; ++j) {
            for (int q = 0; q < TG_NCOUNTERS; ++q) {
                uint64_t x = mix64(key + (uint64_t)(j * TG_NCOUNTERS + q + 1) * GOLDEN);
                double u = (double)(x >> 11) * 0x1.0p-53;
                float v;
                if ((c->nan_mask >> q) & 1u) v = NAN;
                else if (c->nan_frac > 0 && (double)(mix64(x ^ 0xa5a5a5a5ULL) >> 11) * 0x1.0p-53 < c->nan_frac) v = NAN;
                else if (c->counter_dist == 1) v = (float)exp(llo + u * (lhi - llo));
                else v = (float)(lo + u * (hi - lo));
                counters[j * TG_NCOUNTERS + q] = v;
            }
        }
    }
}

void tg_free(tg_trace *t) {
    if (!t) return;
    free(t->k_stream); free(t->k_start); free(t->k_dur); free(t->k_name); free(t->k_layer);
    free(t->r_stream); free(t->r_start); free(t->r_end); free(t->r_depth); free(t->r_op);
    free(t->ncu_name); free(t->class_of_layer); free(t->rep_of_class);
    free(t);
}
