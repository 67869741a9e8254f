/*
 * ucl_oracle.c -- plain, slow, fp64 CPU evaluator of an upper-case-lower-case
 * (UCL) EinSum over tensor-relations.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle that the GPU executor is
 * checked against.  It shares no code, header, table or helper with the GPU
 * path.  Only the test-suite, the smoke check and the CPU-baseline leg of the
 * benchmark may load it; the product path never does.
 *
 * What it computes (paper Sec. 5, Eq. eqn_tr / eqn-TRA and the TR-SQL template
 *   SELECT up(W), SUM(K(valU,valV)) FROM U NATURAL JOIN V GROUP BY up(W)):
 *
 *   1. parse the spec and classify labels (Sec. 4.3: upper-case letters are
 *      promoted to key columns, lower-case letters index the dense tile);
 *   2. natural join of the input relations on every shared upper label
 *      (Sec. 5; with no shared label the join is a cross product, Sec. 7.2);
 *      tuple at a time, with a sorted index on the inner relation;
 *   3. the kernel K: naive loops over every lower-label index combination,
 *      W[lower W] += prod_k U_k[lower U_k], accumulated in fp64, together
 *      with the magnitude sum |prod| used by the parity tolerance;
 *   4. hash group-by on the output key (the projection onto up(W));
 *   5. epilogue after the full sum (scale, optional relu -- the unary
 *      sum-over-empty-set EinSum of Sec. 3's MLP example), then one
 *      round-to-nearest-even cast to the output type;
 *   6. every output key produced by at least one joined tuple is emitted,
 *      in ascending lexicographic order of the key tuple.
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   - one tuple per key (Sec. 4.2: the point lookup "returns a single tuple");
 *     a duplicate key is an error;
 *   - zero-tuple elimination (Sec. 4.2, "can be eliminated") is not applied to
 *     the output: a key produced by the join is kept even if its sum is 0;
 *   - tiles are row-major over the operand's lower-case letters, in the order
 *     they appear in the operand, last letter fastest;
 *   - the extended EinSum of Sec. 3 (Eq. Einsum's general form, an aggregate
 *     ⊕ over the joined values of a scalar function ⊗): ⊕ is SUM, MAX or MIN,
 *     ⊗ is the product (default), sum, difference or quotient of the two
 *     inputs' entries, followed by an element map (identity, relu, exp or
 *     square) -- e.g. Sec. 3's max_j (U_ij - V_ij)^2 is MAX, SUB, SQUARE; a
 *     unary EinSum applies the map to its one input (Sec. 3's MLP example);
 *     three inputs take the product only;
 *   - aggregation ranges over the tuples present (SQL GROUP BY): a tuple
 *     absent from a relation contributes nothing, also under MAX or MIN.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum {
    UO_OK = 0,
    UO_ERR_ARG = 1,
    UO_ERR_SPEC = 2,
    UO_ERR_SHAPE = 3,
    UO_ERR_DUP_KEY = 4,
    UO_ERR_KEY_RANGE = 5,
    UO_ERR_OOM = 6,
    UO_ERR_UNSUPPORTED = 8
};

enum { UO_EPI_NONE = 0, UO_EPI_RELU = 1 };
enum { UO_AGG_SUM = 0, UO_AGG_MAX = 1, UO_AGG_MIN = 2 };
enum { UO_COMB_MUL = 0, UO_COMB_ADD = 1, UO_COMB_SUB = 2, UO_COMB_DIV = 3 };
enum { UO_MAP_IDENT = 0, UO_MAP_RELU = 1, UO_MAP_EXP = 2, UO_MAP_SQUARE = 3 };
enum { UO_OUT_BF16 = 0, UO_OUT_F32 = 1, UO_OUT_F64 = 2 };

#define UO_MAXIN 3
#define UO_MAXLAB 52
#define UO_MAXOPLEN 16

typedef struct {
    int64_t n;             /* number of tuples */
    int u;                 /* number of key columns (upper-case letters) */
    const int32_t *keys;   /* [n, u] row-major */
    const int64_t *bounds; /* [u] key bounds */
    int r;                 /* number of tile dims (lower-case letters) */
    const int64_t *shape;  /* [r] */
    const double *vals;    /* [n, prod(shape)] row-major tiles */
} uo_rel;

typedef struct {
    int epi;
    double scale;
    int out_dtype;
    const int32_t *sample_keys; /* optional [n_sample, uw]: only these groups are evaluated */
    int64_t n_sample;
    int agg, comb, map;         /* extended EinSum: aggregate, combination, element map */
} uo_opts;

typedef struct {
    int64_t m;        /* output tuples */
    int uw, rw;
    int64_t bounds[UO_MAXOPLEN];
    int64_t shape[UO_MAXOPLEN];
    int64_t tile;     /* prod(shape) */
    int32_t *keys;    /* [m, uw] */
    double *acc;      /* [m, tile] raw fp64 sum */
    double *absacc;   /* [m, tile] sum of |terms| (SUM) or largest |term| (MAX, MIN) */
    double *out;      /* [m, tile] after epilogue and cast, stored as double */
    int64_t n_pairs;  /* joined tuples (all of them, also when sampling) */
    int64_t n_mults;  /* n_pairs * prod(all lower extents) */
} uo_result;

/* ---------------------------------------------------------------- parsing */

typedef struct {
    int n_in;
    int len[UO_MAXIN + 1];               /* index n_in = output */
    char op[UO_MAXIN + 1][UO_MAXOPLEN];  /* letters per operand */
    /* per distinct letter */
    int nlab;
    char lab[UO_MAXLAB];
    int upper[UO_MAXLAB];
    int64_t ext[UO_MAXLAB];              /* key bound (upper) or extent (lower) */
    int pos[UO_MAXIN + 1][UO_MAXLAB];    /* key column (upper) or tile dim (lower), -1 if absent */
} uo_spec;

static int is_letter(char c) { return (c >= 'a' && c <= 'z') || (c >= 'A' && c <= 'Z'); }
static int is_up(char c) { return c >= 'A' && c <= 'Z'; }

static int find_lab(const uo_spec *s, char c) {
    for (int i = 0; i < s->nlab; ++i)
        if (s->lab[i] == c) return i;
    return -1;
}

/* Split "op1,op2->out" into operands; every letter is one label, its case
 * fixes whether it is promoted or demoted (Sec. 4.3). */
static int parse_spec(const char *spec, int n_in, uo_spec *s) {
    memset(s, 0, sizeof(*s));
    if (!spec || n_in < 1 || n_in > UO_MAXIN) return UO_ERR_ARG;
    const char *arrow = strstr(spec, "->");
    if (!arrow) return UO_ERR_SPEC;
    int k = 0, l = 0;
    for (const char *p = spec; p < arrow; ++p) {
        if (*p == ',') {
            s->len[k] = l;
            if (++k >= UO_MAXIN) return UO_ERR_SPEC;
            l = 0;
        } else if (is_letter(*p)) {
            if (l >= UO_MAXOPLEN) return UO_ERR_SPEC;
            s->op[k][l++] = *p;
        } else {
            return UO_ERR_SPEC;
        }
    }
    s->len[k] = l;
    if (k + 1 != n_in) return UO_ERR_SPEC;
    s->n_in = n_in;
    l = 0;
    for (const char *p = arrow + 2; *p; ++p) {
        if (!is_letter(*p) || l >= UO_MAXOPLEN) return UO_ERR_SPEC;
        s->op[n_in][l++] = *p;
    }
    s->len[n_in] = l;
    for (int i = 0; i <= n_in; ++i)
        for (int a = 0; a < s->len[i]; ++a)
            for (int b = a + 1; b < s->len[i]; ++b)
                if (s->op[i][a] == s->op[i][b]) return UO_ERR_SPEC; /* repeated label in one operand */
    for (int i = 0; i < n_in; ++i)
        for (int a = 0; a < s->len[i]; ++a) {
            char c = s->op[i][a];
            if (find_lab(s, c) < 0) {
                s->lab[s->nlab] = c;
                s->upper[s->nlab] = is_up(c);
                s->nlab++;
            }
        }
    for (int a = 0; a < s->len[n_in]; ++a)
        if (find_lab(s, s->op[n_in][a]) < 0) return UO_ERR_SPEC; /* output label from nowhere */
    for (int i = 0; i <= n_in; ++i) {
        for (int L = 0; L < s->nlab; ++L) s->pos[i][L] = -1;
        int cu = 0, cl = 0;
        for (int a = 0; a < s->len[i]; ++a) {
            int L = find_lab(s, s->op[i][a]);
            s->pos[i][L] = s->upper[L] ? cu++ : cl++;
        }
    }
    return UO_OK;
}

/* ------------------------------------------------------- relation checks */

static const uo_rel *g_sort_rel;
static const int *g_sort_cols;
static int g_sort_ncols;

static int cmp_by_cols(const void *a, const void *b) {
    int64_t i = *(const int64_t *)a, j = *(const int64_t *)b;
    const uo_rel *R = g_sort_rel;
    for (int c = 0; c < g_sort_ncols; ++c) {
        int32_t x = R->keys[i * R->u + g_sort_cols[c]], y = R->keys[j * R->u + g_sort_cols[c]];
        if (x != y) return x < y ? -1 : 1;
    }
    return (i > j) - (i < j);
}

/* Tuple indices of R sorted by the given key columns (stable on index). */
static int64_t *sorted_index(const uo_rel *R, const int *cols, int ncols) {
    int64_t *idx = (int64_t *)malloc(sizeof(int64_t) * (R->n > 0 ? R->n : 1));
    if (!idx) return NULL;
    for (int64_t i = 0; i < R->n; ++i) idx[i] = i;
    g_sort_rel = R;
    g_sort_cols = cols;
    g_sort_ncols = ncols;
    if (R->n > 1) qsort(idx, (size_t)R->n, sizeof(int64_t), cmp_by_cols);
    return idx;
}

/* Key range and one-tuple-per-key checks (Sec. 4.2). */
static int check_rel(const uo_rel *R) {
    for (int64_t i = 0; i < R->n; ++i)
        for (int c = 0; c < R->u; ++c) {
            int32_t v = R->keys[i * R->u + c];
            if (v < 0 || (int64_t)v >= R->bounds[c]) return UO_ERR_KEY_RANGE;
        }
    if (R->u == 0) return R->n > 1 ? UO_ERR_DUP_KEY : UO_OK;
    int cols[UO_MAXOPLEN];
    for (int c = 0; c < R->u; ++c) cols[c] = c;
    int64_t *idx = sorted_index(R, cols, R->u);
    if (!idx) return UO_ERR_OOM;
    int st = UO_OK;
    for (int64_t i = 1; i < R->n && st == UO_OK; ++i) {
        if (!memcmp(&R->keys[idx[i] * R->u], &R->keys[idx[i - 1] * R->u], sizeof(int32_t) * R->u))
            st = UO_ERR_DUP_KEY;
    }
    free(idx);
    return st;
}

/* ------------------------------------------------------------ group-by map */

typedef struct {
    int uw;
    int64_t cap;      /* power of two */
    int64_t *slot;    /* group id or -1 */
    int64_t ngroups, gcap;
    int32_t *keys;    /* [gcap, uw] */
} uo_map;

static uint64_t hash_key(const int32_t *k, int uw) {
    uint64_t h = 1469598103934665603ULL;
    for (int c = 0; c < uw; ++c) {
        h ^= (uint32_t)k[c];
        h *= 1099511628211ULL;
        h ^= h >> 29;
    }
    return h;
}

static int map_init(uo_map *m, int uw) {
    memset(m, 0, sizeof(*m));
    m->uw = uw;
    m->cap = 1024;
    m->slot = (int64_t *)malloc(sizeof(int64_t) * m->cap);
    m->gcap = 256;
    m->keys = (int32_t *)malloc(sizeof(int32_t) * (size_t)m->gcap * (uw > 0 ? uw : 1));
    if (!m->slot || !m->keys) return UO_ERR_OOM;
    for (int64_t i = 0; i < m->cap; ++i) m->slot[i] = -1;
    return UO_OK;
}

static void map_free(uo_map *m) {
    free(m->slot);
    free(m->keys);
}

static int64_t map_find(const uo_map *m, const int32_t *k) {
    uint64_t h = hash_key(k, m->uw) & (uint64_t)(m->cap - 1);
    while (m->slot[h] >= 0) {
        if (!memcmp(&m->keys[m->slot[h] * m->uw], k, sizeof(int32_t) * m->uw)) return m->slot[h];
        h = (h + 1) & (uint64_t)(m->cap - 1);
    }
    return -1;
}

/* Find or insert; returns the group id, -1 on allocation failure. */
static int64_t map_insert(uo_map *m, const int32_t *k) {
    int64_t g = map_find(m, k);
    if (g >= 0) return g;
    if (2 * (m->ngroups + 1) > m->cap) {
        int64_t ncap = m->cap * 2;
        int64_t *ns = (int64_t *)malloc(sizeof(int64_t) * ncap);
        if (!ns) return -1;
        for (int64_t i = 0; i < ncap; ++i) ns[i] = -1;
        for (int64_t gi = 0; gi < m->ngroups; ++gi) {
            uint64_t h = hash_key(&m->keys[gi * m->uw], m->uw) & (uint64_t)(ncap - 1);
            while (ns[h] >= 0) h = (h + 1) & (uint64_t)(ncap - 1);
            ns[h] = gi;
        }
        free(m->slot);
        m->slot = ns;
        m->cap = ncap;
    }
    if (m->ngroups == m->gcap) {
        int64_t ng = m->gcap * 2;
        int32_t *nk = (int32_t *)realloc(m->keys, sizeof(int32_t) * (size_t)ng * (m->uw > 0 ? m->uw : 1));
        if (!nk) return -1;
        m->keys = nk;
        m->gcap = ng;
    }
    g = m->ngroups++;
    memcpy(&m->keys[g * m->uw], k, sizeof(int32_t) * m->uw);
    uint64_t h = hash_key(k, m->uw) & (uint64_t)(m->cap - 1);
    while (m->slot[h] >= 0) h = (h + 1) & (uint64_t)(m->cap - 1);
    m->slot[h] = g;
    return g;
}

/* ----------------------------------------------------------------- rounding */

/* Round-to-nearest-even of a double to bfloat16 (8 exponent bits, 8
 * significant bits), returned as a double; written from the format's
 * definition: the quantum is 2^(e-8) for |x| in [2^(e-1), 2^e), never finer
 * than the subnormal quantum 2^-133; results at or above 2^128 overflow. */
static double round_bf16(double x) {
    if (x == 0.0 || isnan(x) || isinf(x)) return x;
    int e;
    frexp(x, &e);
    int qe = e - 8;
    if (qe < -133) qe = -133;
    double q = ldexp(1.0, qe);
    double r = nearbyint(x / q) * q; /* default rounding mode: ties to even */
    if (fabs(r) >= ldexp(1.0, 128)) return x > 0 ? INFINITY : -INFINITY;
    return r;
}

static double cast_out(double x, int dt) {
    if (dt == UO_OUT_F32) return (double)(float)x;
    if (dt == UO_OUT_BF16) return round_bf16(x);
    return x;
}

double uo_round_bf16(double x) { return round_bf16(x); }

/* ------------------------------------------------------------------ einsum */

typedef struct {
    const uo_spec *s;
    const uo_rel *rel;
    uo_opts opts;
    /* join indices: per level k >= 1, the columns of rel k shared with rels < k */
    int nshared[UO_MAXIN];
    int shared_lab[UO_MAXIN][UO_MAXOPLEN];
    int shared_col[UO_MAXIN][UO_MAXOPLEN];
    int64_t *index[UO_MAXIN];
    /* current binding of upper labels */
    int32_t bind[UO_MAXLAB];
    int64_t tup[UO_MAXIN];
    /* lower loop nest: all lower labels, strides per input and in W */
    int nlow;
    int64_t lext[UO_MAXLAB];
    int64_t lstr[UO_MAXIN + 1][UO_MAXLAB];
    int64_t tile_in[UO_MAXIN];
    int64_t tile_w;
    /* output */
    uo_map groups;
    uo_map sample;
    int use_sample;
    double *acc, *absacc;
    int64_t acc_cap;
    int64_t n_pairs;
    int err;
} uo_ctx;

/* One term of the extended EinSum: the combination of the joined entries,
 * then the element map. */
static double term(const uo_opts *o, int n_in, const double *x) {
    double p;
    if (n_in == 1) {
        p = x[0];
    } else if (n_in == 3 || o->comb == UO_COMB_MUL) {
        p = 1.0;
        for (int k = 0; k < n_in; ++k) p *= x[k];
    } else if (o->comb == UO_COMB_ADD) {
        p = x[0] + x[1];
    } else if (o->comb == UO_COMB_SUB) {
        p = x[0] - x[1];
    } else {
        p = x[0] / x[1];
    }
    switch (o->map) {
        case UO_MAP_RELU: return p > 0 ? p : 0.0;
        case UO_MAP_EXP: return exp(p);
        case UO_MAP_SQUARE: return p * p;
        default: return p;
    }
}

/* Fold one term into the aggregate and its magnitude bound. */
static void fold(const uo_opts *o, double *acc, double *absv, double p) {
    if (o->agg == UO_AGG_MAX) {
        if (p > *acc) *acc = p;
        if (fabs(p) > *absv) *absv = fabs(p);
    } else if (o->agg == UO_AGG_MIN) {
        if (p < *acc) *acc = p;
        if (fabs(p) > *absv) *absv = fabs(p);
    } else {
        *acc += p;
        *absv += fabs(p);
    }
}

/* Kernel K for one joined tuple (Sec. 5): naive loop over every lower-label
 * index combination, W[...] ⊕= ⊗_k U_k[...]; the last lower label is the
 * innermost loop. */
static void apply_kernel(uo_ctx *c, int64_t g) {
    const uo_spec *s = c->s;
    const double *base[UO_MAXIN];
    for (int k = 0; k < s->n_in; ++k) base[k] = c->rel[k].vals + c->tup[k] * c->tile_in[k];
    double *accg = c->acc + g * c->tile_w;
    double *absg = c->absacc + g * c->tile_w;
    int64_t idx[UO_MAXLAB];
    for (int L = 0; L < c->nlow; ++L) idx[L] = 0;
    double x[UO_MAXIN];
    if (c->nlow == 0) {
        for (int k = 0; k < s->n_in; ++k) x[k] = base[k][0];
        fold(&c->opts, &accg[0], &absg[0], term(&c->opts, s->n_in, x));
        return;
    }
    int last = c->nlow - 1;
    for (;;) {
        int64_t off[UO_MAXIN + 1] = {0, 0, 0, 0};
        for (int L = 0; L < last; ++L)
            for (int k = 0; k <= s->n_in; ++k) off[k] += idx[L] * c->lstr[k][L];
        for (int64_t t = 0; t < c->lext[last]; ++t) {
            for (int k = 0; k < s->n_in; ++k) x[k] = base[k][off[k] + t * c->lstr[k][last]];
            int64_t w = off[s->n_in] + t * c->lstr[s->n_in][last];
            fold(&c->opts, &accg[w], &absg[w], term(&c->opts, s->n_in, x));
        }
        int L = last - 1;
        while (L >= 0) {
            if (++idx[L] < c->lext[L]) break;
            idx[L] = 0;
            --L;
        }
        if (L < 0) break;
    }
}

/* A fully joined tuple: project onto up(W), group, run the kernel. */
static void emit_joined(uo_ctx *c) {
    const uo_spec *s = c->s;
    int n = s->n_in;
    int32_t key[UO_MAXOPLEN];
    int uw = 0;
    for (int a = 0; a < s->len[n]; ++a) {
        int L = find_lab(s, s->op[n][a]);
        if (s->upper[L]) key[uw++] = c->bind[L];
    }
    c->n_pairs++;
    if (c->use_sample && map_find(&c->sample, key) < 0) return;
    int64_t g = map_insert(&c->groups, key);
    if (g < 0) {
        c->err = UO_ERR_OOM;
        return;
    }
    if (g >= c->acc_cap) {
        int64_t ncap = c->acc_cap ? c->acc_cap * 2 : 64;
        while (ncap <= g) ncap *= 2;
        double *na = (double *)realloc(c->acc, sizeof(double) * (size_t)(ncap * c->tile_w));
        if (!na) { c->err = UO_ERR_OOM; return; }
        c->acc = na;
        double *nb = (double *)realloc(c->absacc, sizeof(double) * (size_t)(ncap * c->tile_w));
        if (!nb) { c->err = UO_ERR_OOM; return; }
        c->absacc = nb;
        /* the aggregate's identity: 0, or -inf / +inf for MAX / MIN (replaced
           by the first term, as every joined tuple reaches every entry) */
        const double id = c->opts.agg == UO_AGG_MAX ? -INFINITY : (c->opts.agg == UO_AGG_MIN ? INFINITY : 0.0);
        for (int64_t i = c->acc_cap * c->tile_w; i < ncap * c->tile_w; ++i) c->acc[i] = id;
        memset(c->absacc + c->acc_cap * c->tile_w, 0, sizeof(double) * (size_t)((ncap - c->acc_cap) * c->tile_w));
        c->acc_cap = ncap;
    }
    apply_kernel(c, g);
}

/* Natural join, one relation per level, tuple at a time (Sec. 5): at level k
 * the candidates are the tuples of rel k whose shared upper labels equal the
 * current binding, found by binary search in rel k's sorted index. */
static void join_level(uo_ctx *c, int k) {
    if (c->err) return;
    const uo_spec *s = c->s;
    if (k == s->n_in) {
        emit_joined(c);
        return;
    }
    const uo_rel *R = &c->rel[k];
    int64_t lo = 0, hi = R->n;
    const int64_t *ix = c->index[k];
    if (c->nshared[k] > 0) {
        /* lower bound */
        int64_t a = 0, b = R->n;
        while (a < b) {
            int64_t mid = (a + b) / 2;
            int cmp = 0;
            for (int q = 0; q < c->nshared[k] && !cmp; ++q) {
                int32_t x = R->keys[ix[mid] * R->u + c->shared_col[k][q]];
                int32_t y = c->bind[c->shared_lab[k][q]];
                cmp = (x > y) - (x < y);
            }
            if (cmp < 0) a = mid + 1; else b = mid;
        }
        lo = a;
        b = R->n;
        while (a < b) {
            int64_t mid = (a + b) / 2;
            int cmp = 0;
            for (int q = 0; q < c->nshared[k] && !cmp; ++q) {
                int32_t x = R->keys[ix[mid] * R->u + c->shared_col[k][q]];
                int32_t y = c->bind[c->shared_lab[k][q]];
                cmp = (x > y) - (x < y);
            }
            if (cmp <= 0) a = mid + 1; else b = mid;
        }
        hi = a;
    }
    for (int64_t t = lo; t < hi && !c->err; ++t) {
        int64_t i = ix[t];
        c->tup[k] = i;
        for (int L = 0; L < s->nlab; ++L)
            if (s->upper[L] && s->pos[k][L] >= 0) c->bind[L] = R->keys[i * R->u + s->pos[k][L]];
        join_level(c, k + 1);
    }
}

static const int32_t *g_out_keys;
static int g_out_uw;
static int cmp_group(const void *a, const void *b) {
    int64_t i = *(const int64_t *)a, j = *(const int64_t *)b;
    for (int q = 0; q < g_out_uw; ++q) {
        int32_t x = g_out_keys[i * g_out_uw + q], y = g_out_keys[j * g_out_uw + q];
        if (x != y) return x < y ? -1 : 1;
    }
    return 0;
}

void uo_free(uo_result *r) {
    if (!r) return;
    free(r->keys);
    free(r->acc);
    free(r->absacc);
    free(r->out);
    memset(r, 0, sizeof(*r));
}

int uo_einsum(const char *spec, int n_in, const uo_rel *rels, const uo_opts *opts, uo_result *res) {
    if (!res || !rels) return UO_ERR_ARG;
    memset(res, 0, sizeof(*res));
    uo_spec s;
    int st = parse_spec(spec, n_in, &s);
    if (st) return st;
    if (opts && opts->epi != UO_EPI_NONE && opts->epi != UO_EPI_RELU) return UO_ERR_ARG;
    if (opts && (opts->out_dtype < UO_OUT_BF16 || opts->out_dtype > UO_OUT_F64)) return UO_ERR_ARG;
    if (opts && (opts->agg < UO_AGG_SUM || opts->agg > UO_AGG_MIN || opts->comb < UO_COMB_MUL ||
                 opts->comb > UO_COMB_DIV || opts->map < UO_MAP_IDENT || opts->map > UO_MAP_SQUARE))
        return UO_ERR_ARG;
    if (opts && n_in == 3 && (opts->agg != UO_AGG_SUM || opts->comb != UO_COMB_MUL || opts->map != UO_MAP_IDENT))
        return UO_ERR_UNSUPPORTED;

    /* arity and extents: one bound / extent per label across all operands (Sec. 3 bounds) */
    for (int k = 0; k < n_in; ++k) {
        const uo_rel *R = &rels[k];
        int nu = 0, nl = 0;
        for (int a = 0; a < s.len[k]; ++a) {
            if (is_up(s.op[k][a])) nu++;
            else nl++;
        }
        if (R->n < 0 || R->u != nu || R->r != nl) return UO_ERR_SHAPE;
        if (R->n > 0 && ((R->u > 0 && !R->keys) || !R->vals)) return UO_ERR_ARG;
        for (int L = 0; L < s.nlab; ++L) {
            int p = s.pos[k][L];
            if (p < 0) continue;
            int64_t e = s.upper[L] ? R->bounds[p] : R->shape[p];
            if (e < 1) return UO_ERR_SHAPE;
            if (s.ext[L] == 0) s.ext[L] = e;
            else if (s.ext[L] != e) return UO_ERR_SHAPE;
        }
    }
    for (int k = 0; k < n_in; ++k) {
        st = check_rel(&rels[k]);
        if (st) return st;
    }

    uo_ctx c;
    memset(&c, 0, sizeof(c));
    c.s = &s;
    c.rel = rels;
    c.opts.epi = UO_EPI_NONE;
    c.opts.scale = 1.0;
    c.opts.out_dtype = UO_OUT_F64;
    if (opts) c.opts = *opts;

    /* output shape */
    int uw = 0, rw = 0;
    for (int a = 0; a < s.len[n_in]; ++a) {
        int L = find_lab(&s, s.op[n_in][a]);
        if (s.upper[L]) res->bounds[uw++] = s.ext[L];
        else res->shape[rw++] = s.ext[L];
    }
    res->uw = uw;
    res->rw = rw;

    /* lower loop nest */
    c.tile_w = 1;
    for (int q = 0; q < rw; ++q) c.tile_w *= res->shape[q];
    res->tile = c.tile_w;
    for (int k = 0; k < n_in; ++k) {
        c.tile_in[k] = 1;
        for (int q = 0; q < rels[k].r; ++q) c.tile_in[k] *= rels[k].shape[q];
    }
    int64_t low_prod = 1;
    for (int L = 0; L < s.nlab; ++L) {
        if (s.upper[L]) continue;
        int j = c.nlow++;
        c.lext[j] = s.ext[L];
        low_prod *= s.ext[L];
        for (int k = 0; k <= n_in; ++k) {
            /* row-major stride of label L in operand k's tile (0 if absent) */
            int64_t str = 0;
            int p = s.pos[k][L];
            if (p >= 0) {
                str = 1;
                for (int a = s.len[k] - 1; a >= 0; --a) {
                    int L2 = find_lab(&s, s.op[k][a]);
                    if (s.upper[L2]) continue;
                    if (s.pos[k][L2] == p) break;
                    str *= s.ext[L2];
                }
            }
            c.lstr[k][j] = str;
        }
    }

    /* sorted indices for the index nested loop join */
    for (int k = 0; k < n_in; ++k) {
        int cols[UO_MAXOPLEN];
        c.nshared[k] = 0;
        for (int L = 0; L < s.nlab; ++L) {
            if (!s.upper[L] || s.pos[k][L] < 0) continue;
            int seen = 0;
            for (int k2 = 0; k2 < k; ++k2) seen |= s.pos[k2][L] >= 0;
            if (!seen) continue;
            c.shared_lab[k][c.nshared[k]] = L;
            c.shared_col[k][c.nshared[k]] = s.pos[k][L];
            cols[c.nshared[k]] = s.pos[k][L];
            c.nshared[k]++;
        }
        c.index[k] = sorted_index(&rels[k], cols, c.nshared[k]);
        if (!c.index[k]) { st = UO_ERR_OOM; goto done; }
    }

    st = map_init(&c.groups, uw);
    if (st) goto done;
    if (c.opts.sample_keys && c.opts.n_sample >= 0) {
        c.use_sample = 1;
        st = map_init(&c.sample, uw);
        if (st) goto done;
        for (int64_t i = 0; i < c.opts.n_sample; ++i)
            if (map_insert(&c.sample, &c.opts.sample_keys[i * uw]) < 0) { st = UO_ERR_OOM; goto done; }
    }

    join_level(&c, 0);
    if (c.err) { st = c.err; goto done; }

    /* emit groups in ascending key order, epilogue then one cast */
    {
        int64_t m = c.groups.ngroups;
        int64_t *order = (int64_t *)malloc(sizeof(int64_t) * (m > 0 ? m : 1));
        res->keys = (int32_t *)malloc(sizeof(int32_t) * (size_t)(m > 0 ? m : 1) * (uw > 0 ? uw : 1));
        res->acc = (double *)malloc(sizeof(double) * (size_t)((m > 0 ? m : 1) * c.tile_w));
        res->absacc = (double *)malloc(sizeof(double) * (size_t)((m > 0 ? m : 1) * c.tile_w));
        res->out = (double *)malloc(sizeof(double) * (size_t)((m > 0 ? m : 1) * c.tile_w));
        if (!order || !res->keys || !res->acc || !res->absacc || !res->out) {
            free(order);
            uo_free(res);
            st = UO_ERR_OOM;
            goto done;
        }
        for (int64_t i = 0; i < m; ++i) order[i] = i;
        g_out_keys = c.groups.keys;
        g_out_uw = uw;
        if (m > 1 && uw > 0) qsort(order, (size_t)m, sizeof(int64_t), cmp_group);
        for (int64_t i = 0; i < m; ++i) {
            int64_t g = order[i];
            memcpy(&res->keys[i * uw], &c.groups.keys[g * uw], sizeof(int32_t) * uw);
            for (int64_t w = 0; w < c.tile_w; ++w) {
                double a = c.acc[g * c.tile_w + w];
                res->acc[i * c.tile_w + w] = a;
                res->absacc[i * c.tile_w + w] = c.absacc[g * c.tile_w + w];
                double o = c.opts.scale * a;
                if (c.opts.epi == UO_EPI_RELU && o < 0) o = 0.0;
                res->out[i * c.tile_w + w] = cast_out(o, c.opts.out_dtype);
            }
        }
        free(order);
        res->m = m;
        res->n_pairs = c.n_pairs;
        res->n_mults = c.n_pairs * low_prod;
    }

done:
    for (int k = 0; k < n_in; ++k) free(c.index[k]);
    map_free(&c.groups);
    if (c.use_sample) map_free(&c.sample);
    free(c.acc);
    free(c.absacc);
    return st;
}
