/*
 * Plain CPU oracle for eager multi-resolution substrate discovery (float64).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may call, link or
 * load this file: only the tests, the smoke check and the benchmark's CPU
 * baseline leg use it. It shares no code, header, table or constant with the
 * CUDA library; it is deliberately slow and written to be checked by eye
 * against the paper:
 *
 *   - grid:   Eq. 1 (Section 3.1), Grid_d = {((2i+1)/2^{d+1} - 1, (2j+1)/2^{d+1} - 1)}
 *             for i, j in [0, 2^{d+1}), d = 0..D; N_total = (4^{D+2} - 4) / 3.
 *   - query:  W = CPPN(s, T) over every grid position (Section 3.1); a CPPN maps
 *             (x1, y1, x2, y2) to a weight (Section 2); the fifth input is the
 *             bias, fixed at 1.
 *   - filter: variance computed bottom-up from each cell's four children, the
 *             active mask of Eq. 2 propagated top-down (Section 3.2), and the
 *             ES-HyperNEAT band test with threshold theta_band (Theorem 1 and
 *             Section 3.3 name it; the rule itself is ES-HyperNEAT's).
 *   - lazy:   the sequential ES-HyperNEAT quadtree of Fig. 1 (left) and
 *             Section 2, used to check Theorem 1 (lazy subset of eager).
 *
 * Readings where the paper is silent (each one is listed with its reason in
 * the design notes): variance over the 4 children with ddof 0; a cell at the
 * maximum depth is a leaf (never split); band neighbours at the Grid_d
 * spacing 2^-d, evaluated outside [-1,1]^2 when the cell is on the border;
 * one threshold theta for both division and extraction; strict comparisons
 * (V > theta splits, B > band passes, |w| > w_min passes when w_min > 0);
 * activations sigmoid 1/(1+e^-z), tanh, gauss e^(-z^2), sin, |z|, identity
 * with no scaling; a node's pre-activation is bias + sum of w * source value
 * over its enabled in-connections.
 *
 * Positions are numbered depth-major: global index = off(d) + m with
 * off(d) = (4^{d+1} - 4) / 3 and m the Morton code of (i, j) (bit k of i to
 * bit 2k, bit k of j to bit 2k+1). Halo points (the out-of-domain band
 * neighbours) of depth d are numbered hoff(d) + side * 2^{d+1} + t with
 * hoff(d) = 8 (2^d - 1); side 0: (i=-1, j=t), 1: (i=2^{d+1}, j=t),
 * 2: (i=t, j=-1), 3: (i=t, j=2^{d+1}).
 *
 * Each decision also carries a forward error bound for the fp32 evaluation
 * the device performs (standard rounding-error analysis: a k-term sum
 * carries at most gamma_k = k u / (1 - k u) times the sum of magnitudes,
 * u = 2^-24; activations are Lipschitz; the device's activations are allowed
 * a fixed absolute error, checked separately against the device). A decision
 * whose margin to its threshold is within 1e-6 plus its bound is reported as
 * uncertain; the parity tests count those and skip them.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORA_OK 0
#define ORA_ERR_ARG 1
#define ORA_ERR_CYCLE 2
#define ORA_ERR_ALLOC 3

#define KIND_HIDDEN 5
#define KIND_OUTPUT 6
#define MAX_DEPTH 14

static const double U32 = 5.9604644775390625e-08; /* 2^-24, fp32 unit roundoff */
static const double ACT_ABS_BUDGET = 9.5367431640625e-07; /* 2^-20 */
static const double SIN_ABS_BUDGET = 1.9073486328125e-06; /* 2^-19 */
static const double SIN_ARG_LIMIT = 8192.0;
static const double TIE_MARGIN = 1e-6;

static double gamma_n(int n) { return n * U32 / (1.0 - n * U32); }

/* ---- activations (fp64) ------------------------------------------------ */

static double act_value(int a, double z)
{
    switch (a) {
    case 0: return z;
    case 1: return 1.0 / (1.0 + exp(-z));
    case 2: return tanh(z);
    case 3: return exp(-z * z);
    case 4: return sin(z);
    case 5: return fabs(z);
    default: return NAN;
    }
}

/* Lipschitz constant of each activation over the reals. gauss: max |d/dz e^{-z^2}|
 * = sqrt(2/e) at z = 1/sqrt(2). */
static double act_lipschitz(int a)
{
    switch (a) {
    case 1: return 0.25;
    case 3: return 0.85776388496070679648;
    default: return 1.0;
    }
}

/* Absolute error allowed to the device's fp32 activation at input z. */
static double act_budget(int a, double z, double v)
{
    switch (a) {
    case 0: case 5: return 0.0;
    case 1: case 2: case 3: return ACT_ABS_BUDGET + U32 * fabs(v);
    case 4: return fabs(z) <= SIN_ARG_LIMIT ? SIN_ABS_BUDGET + U32 * fabs(v) : INFINITY;
    default: return INFINITY;
    }
}

/* ---- genome preparation: ids -> local indices, Kahn topological order ----- */

typedef struct {
    int n;             /* nodes */
    int out;           /* local index of the output node */
    const int32_t *kind, *act;
    const float *bias;
    int *order;        /* [n] topological order of local indices */
    int *in_beg, *in_cnt; /* [n] in-edge ranges into src/w */
    int *src;          /* [ne] local source index */
    double *w;         /* [ne] */
} genome_t;

static void genome_free(genome_t *G)
{
    free(G->order); free(G->in_beg); free(G->in_cnt); free(G->src); free(G->w);
    memset(G, 0, sizeof *G);
}

static int local_of(const int32_t *ids, int n, int32_t id)
{
    for (int k = 0; k < n; k++)
        if (ids[k] == id) return k;
    return -1;
}

/* Build genome g. Returns ORA_OK, ORA_ERR_ARG (bad ids, no/duplicate output,
 * connection into an input) or ORA_ERR_CYCLE (the enabled connections are not
 * acyclic: Kahn's algorithm cannot order every node). */
static int genome_build(genome_t *G, int g, const int64_t *node_ptr, const int32_t *node_id,
                        const int32_t *node_kind, const int32_t *node_act, const float *node_bias,
                        const int64_t *conn_ptr, const int32_t *conn_src, const int32_t *conn_dst,
                        const float *conn_w, const uint8_t *conn_en)
{
    memset(G, 0, sizeof *G);
    int64_t n0 = node_ptr[g], n1 = node_ptr[g + 1], c0 = conn_ptr[g], c1 = conn_ptr[g + 1];
    int n = (int)(n1 - n0);
    if (n <= 0) return ORA_ERR_ARG;
    const int32_t *ids = node_id + n0;
    G->n = n;
    G->kind = node_kind + n0;
    G->act = node_act + n0;
    G->bias = node_bias + n0;
    G->out = -1;
    for (int k = 0; k < n; k++) {
        if (G->kind[k] < 0 || G->kind[k] > KIND_OUTPUT) return ORA_ERR_ARG;
        if (G->kind[k] >= KIND_HIDDEN && (G->act[k] < 0 || G->act[k] > 5)) return ORA_ERR_ARG;
        if (local_of(ids, k, ids[k]) >= 0) return ORA_ERR_ARG; /* duplicate id */
        if (G->kind[k] == KIND_OUTPUT) {
            if (G->out >= 0) return ORA_ERR_ARG;
            G->out = k;
        }
    }
    if (G->out < 0) return ORA_ERR_ARG;
    int ne = 0;
    for (int64_t c = c0; c < c1; c++) ne += conn_en[c] ? 1 : 0;
    int *esrc = malloc(sizeof(int) * (ne + 1)), *edst = malloc(sizeof(int) * (ne + 1));
    double *ew = malloc(sizeof(double) * (ne + 1));
    G->order = malloc(sizeof(int) * n);
    G->in_beg = calloc(n, sizeof(int));
    G->in_cnt = calloc(n, sizeof(int));
    G->src = malloc(sizeof(int) * (ne + 1));
    G->w = malloc(sizeof(double) * (ne + 1));
    int *indeg = calloc(n, sizeof(int));
    char *done = calloc(n, 1);
    if (!esrc || !edst || !ew || !G->order || !G->in_beg || !G->in_cnt || !G->src || !G->w || !indeg || !done) {
        free(esrc); free(edst); free(ew); free(indeg); free(done); genome_free(G);
        return ORA_ERR_ALLOC;
    }
    int k = 0, rc = ORA_OK;
    for (int64_t c = c0; c < c1 && rc == ORA_OK; c++) {
        if (!conn_en[c]) continue;
        int s = local_of(ids, n, conn_src[c]), d = local_of(ids, n, conn_dst[c]);
        if (s < 0 || d < 0 || G->kind[d] < KIND_HIDDEN) rc = ORA_ERR_ARG;
        esrc[k] = s; edst[k] = d; ew[k] = (double)conn_w[c]; k++;
    }
    if (rc == ORA_OK) {
        /* group in-edges by destination, keeping the connection order */
        for (int e = 0; e < ne; e++) G->in_cnt[edst[e]]++;
        for (int v = 1; v < n; v++) G->in_beg[v] = G->in_beg[v - 1] + G->in_cnt[v - 1];
        int *fill = calloc(n, sizeof(int));
        for (int e = 0; e < ne; e++) {
            int d = edst[e], at = G->in_beg[d] + fill[d]++;
            G->src[at] = esrc[e];
            G->w[at] = ew[e];
            indeg[d]++;
        }
        free(fill);
        /* Kahn's algorithm; among ready nodes the smallest id goes first */
        for (int placed = 0; placed < n; placed++) {
            int pick = -1;
            for (int v = 0; v < n; v++)
                if (!done[v] && indeg[v] == 0 && (pick < 0 || ids[v] < ids[pick])) pick = v;
            if (pick < 0) { rc = ORA_ERR_CYCLE; break; }
            done[pick] = 1;
            G->order[placed] = pick;
            for (int e = 0; e < ne; e++)
                if (esrc[e] == pick) indeg[edst[e]]--;
        }
    }
    free(esrc); free(edst); free(ew); free(indeg); free(done);
    if (rc != ORA_OK) genome_free(G);
    return rc;
}

/* ---- CPPN evaluation with an fp32 error bound ----------------------------- */

/* val/err: caller scratch of G->n doubles. in[5] = (x1, y1, x2, y2, bias=1).
 * Each non-input node, in topological order: z = bias + sum w * v_src over its
 * enabled in-connections, v = act(z). err bounds |fp32 result - fp64 result|. */
static double cppn_eval(const genome_t *G, const double in[5], double *val, double *err, double *out_err)
{
    for (int t = 0; t < G->n; t++) {
        int v = G->order[t];
        int kd = G->kind[v];
        if (kd < KIND_HIDDEN) {
            val[v] = in[kd];
            err[v] = 0.0;
            continue;
        }
        double z = (double)G->bias[v];
        double mag = fabs(z), dz = 0.0;
        for (int e = G->in_beg[v]; e < G->in_beg[v] + G->in_cnt[v]; e++) {
            int s = G->src[e];
            z += G->w[e] * val[s];
            mag += fabs(G->w[e]) * (fabs(val[s]) + err[s]);
            dz += fabs(G->w[e]) * err[s];
        }
        /* terms: bias, each edge, plus folded-constant regrouping on the device */
        dz += gamma_n(G->in_cnt[v] + 2) * mag;
        int a = G->act[v];
        val[v] = act_value(a, z);
        err[v] = act_lipschitz(a) * dz + act_budget(a, z, val[v]);
        if (!(err[v] >= 0.0)) err[v] = INFINITY; /* NaN guard */
    }
    *out_err = err[G->out];
    return val[G->out];
}

/* ---- grid: Eq. 1, depth-major Morton numbering ---------------------------- */

static int64_t level_offset(int d) { return (((int64_t)1 << (2 * (d + 1))) - 4) / 3; }
static int64_t halo_offset(int d) { return 8 * (((int64_t)1 << d) - 1); }
static int64_t side_len(int d) { return (int64_t)1 << (d + 1); }

static int64_t morton(int64_t i, int64_t j)
{
    int64_t m = 0;
    for (int k = 0; k < 31; k++) {
        m |= ((i >> k) & 1) << (2 * k);
        m |= ((j >> k) & 1) << (2 * k + 1);
    }
    return m;
}

/* coordinate of grid index i at depth d (i may be -1 or 2^{d+1} for halo points) */
static double coord(int d, int64_t i) { return (2.0 * (double)i + 1.0) / (double)side_len(d) - 1.0; }

static void query_inputs(int side, double a, double b, double x, double y, double in[5])
{
    if (side == 0) { in[0] = a; in[1] = b; in[2] = x; in[3] = y; }
    else { in[0] = x; in[1] = y; in[2] = a; in[3] = b; }
    in[4] = 1.0;
}

/* ---- 3-valued decisions: 0 false, 1 true, 2 uncertain --------------------- */

static int decide_gt(double v, double thr, double margin)
{
    if (!(fabs(v - thr) > margin)) return 2; /* also NaN/inf margins */
    return v > thr ? 1 : 0;
}
static int and3(int a, int b)
{
    if (a == 0 || b == 0) return 0;
    if (a == 1 && b == 1) return 1;
    return 2;
}
static int not3(int a) { return a == 2 ? 2 : 1 - a; }

/* ---- public entry points ------------------------------------------------- */

int ora_version(void) { return 1; }

int64_t ora_n_total(int D) { return level_offset(D + 1); }
int64_t ora_n_halo(int D) { return halo_offset(D + 1); }

/* global index of grid point (d, i, j) */
int64_t ora_index(int d, int64_t i, int64_t j) { return level_offset(d) + morton(i, j); }

/* Check every genome of a population: 0 ok, else ORA_ERR_* of the first bad one in *bad. */
int ora_check_population(int P, const int64_t *node_ptr, const int32_t *node_id, const int32_t *node_kind,
                         const int32_t *node_act, const float *node_bias, const int64_t *conn_ptr,
                         const int32_t *conn_src, const int32_t *conn_dst, const float *conn_w,
                         const uint8_t *conn_en, int32_t *bad)
{
    for (int g = 0; g < P; g++) {
        genome_t G;
        int rc = genome_build(&G, g, node_ptr, node_id, node_kind, node_act, node_bias, conn_ptr,
                              conn_src, conn_dst, conn_w, conn_en);
        if (rc != ORA_OK) { *bad = g; return rc; }
        genome_free(&G);
    }
    *bad = -1;
    return ORA_OK;
}

/* Evaluate genome g at n input vectors in[n][5]; out[n], err[n] (err may be NULL). */
int ora_cppn(int g, const int64_t *node_ptr, const int32_t *node_id, const int32_t *node_kind,
             const int32_t *node_act, const float *node_bias, const int64_t *conn_ptr, const int32_t *conn_src,
             const int32_t *conn_dst, const float *conn_w, const uint8_t *conn_en,
             int64_t n, const double *in, double *out, double *err)
{
    genome_t G;
    int rc = genome_build(&G, g, node_ptr, node_id, node_kind, node_act, node_bias, conn_ptr, conn_src,
                          conn_dst, conn_w, conn_en);
    if (rc != ORA_OK) return rc;
    double *val = malloc(sizeof(double) * G.n), *er = malloc(sizeof(double) * G.n);
    for (int64_t k = 0; k < n; k++) {
        double e;
        out[k] = cppn_eval(&G, in + 5 * k, val, er, &e);
        if (err) err[k] = e;
    }
    free(val); free(er);
    genome_free(&G);
    return ORA_OK;
}

/*
 * Eager discovery for genomes [g0, g1) and S query slots, by definition.
 * Sources: src_a/src_b/src_side are [S] (per_genome = 0) or [P][S] (per_genome = 1);
 * src_count (optional, per-genome mode) limits the slots of genome g.
 * Per (g, s) pair r = (g - g0) * S + s, every output array below that is not
 * NULL holds that pair's values at [r * N_total + global index] (halo arrays:
 * [r * N_halo + halo index]):
 *   w, w_err           CPPN output and its fp32 error bound
 *   w_halo, halo_err   the same at halo points
 *   var, var_err       V(p): variance of p's 4 children (0 at depth D)
 *   bnd, bnd_err       B(p): the band value
 *   keep_eager         fp64 decision of the eager filter (0/1)
 *   unc_eager          1 when that decision is within its margin (uncertain)
 *   keep_gated, unc_gated   the same with Eq. 2's active mask
 *   split              fp64 decision V(p) > theta at depth < D (0/1)
 */
int ora_discover(const int64_t *node_ptr, const int32_t *node_id, const int32_t *node_kind,
                 const int32_t *node_act, const float *node_bias, const int64_t *conn_ptr,
                 const int32_t *conn_src, const int32_t *conn_dst, const float *conn_w, const uint8_t *conn_en,
                 int g0, int g1, int S, const float *src_a, const float *src_b, const int32_t *src_side,
                 int per_genome, const int32_t *src_count,
                 int D, double theta, double band, double w_min,
                 double *w, double *w_err, double *w_halo, double *halo_err,
                 double *var, double *var_err, double *bnd, double *bnd_err,
                 uint8_t *keep_eager, uint8_t *unc_eager, uint8_t *keep_gated, uint8_t *unc_gated,
                 uint8_t *split, int nthreads)
{
    if (D < 0 || D > MAX_DEPTH || g1 < g0 || S < 0) return ORA_ERR_ARG;
    int G = g1 - g0;
    genome_t *gen = calloc(G > 0 ? G : 1, sizeof(genome_t));
    if (!gen) return ORA_ERR_ALLOC;
    int rc = ORA_OK;
    for (int k = 0; k < G && rc == ORA_OK; k++)
        rc = genome_build(&gen[k], g0 + k, node_ptr, node_id, node_kind, node_act, node_bias, conn_ptr,
                          conn_src, conn_dst, conn_w, conn_en);
    if (rc != ORA_OK) {
        for (int k = 0; k < G; k++) genome_free(&gen[k]);
        free(gen);
        return rc;
    }
    const int64_t NT = level_offset(D + 1), NH = halo_offset(D + 1);
    int64_t pairs = (int64_t)G * S;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel
#endif
    {
        double *pw = malloc(sizeof(double) * NT), *pe = malloc(sizeof(double) * NT);
        double *ph = malloc(sizeof(double) * (NH + 1)), *phe = malloc(sizeof(double) * (NH + 1));
        double *pv = malloc(sizeof(double) * NT), *pve = malloc(sizeof(double) * NT);
        uint8_t *act64 = malloc(NT), *act3 = malloc(NT);
        int nmax = 1;
        for (int k = 0; k < G; k++) nmax = gen[k].n > nmax ? gen[k].n : nmax;
        double *val = malloc(sizeof(double) * nmax), *er = malloc(sizeof(double) * nmax);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
        for (int64_t r = 0; r < pairs; r++) {
            int gl = (int)(r / S), s = (int)(r % S), g = g0 + gl;
            const genome_t *Gn = &gen[gl];
            if (per_genome && src_count && s >= src_count[g]) continue;
            int64_t si = per_genome ? (int64_t)g * S + s : s;
            double a = (double)src_a[si], b = (double)src_b[si];
            int side = src_side[si];
            double in[5];
            /* 1. CPPN at every grid position (Eq. 1) and every halo point */
            for (int d = 0; d <= D; d++) {
                int64_t n = side_len(d);
                for (int64_t i = 0; i < n; i++)
                    for (int64_t j = 0; j < n; j++) {
                        int64_t p = level_offset(d) + morton(i, j);
                        query_inputs(side, a, b, coord(d, i), coord(d, j), in);
                        pw[p] = cppn_eval(Gn, in, val, er, &pe[p]);
                    }
                for (int sd = 0; sd < 4; sd++)
                    for (int64_t t = 0; t < n; t++) {
                        int64_t hi = sd == 0 ? -1 : sd == 1 ? n : t;
                        int64_t hj = sd == 2 ? -1 : sd == 3 ? n : t;
                        int64_t h = halo_offset(d) + sd * n + t;
                        query_inputs(side, a, b, coord(d, hi), coord(d, hj), in);
                        ph[h] = cppn_eval(Gn, in, val, er, &phe[h]);
                    }
            }
            /* 2. variance of each cell's four children, bottom-up (Section 3.2) */
            for (int d = 0; d <= D; d++) {
                int64_t n = side_len(d);
                for (int64_t i = 0; i < n; i++)
                    for (int64_t j = 0; j < n; j++) {
                        int64_t p = level_offset(d) + morton(i, j);
                        if (d == D) { pv[p] = 0.0; pve[p] = 0.0; continue; }
                        double c[4], ce[4], m = 0.0, me = 0.0, cm = 0.0;
                        for (int q = 0; q < 4; q++) {
                            int64_t ch = level_offset(d + 1) + morton(2 * i + (q & 1), 2 * j + (q >> 1));
                            c[q] = pw[ch]; ce[q] = pe[ch];
                            m += c[q] / 4.0; me += ce[q] / 4.0; cm += fabs(c[q]) / 4.0;
                        }
                        me += gamma_n(4) * cm;
                        double v = 0.0, ve = 0.0;
                        for (int q = 0; q < 4; q++) {
                            double dq = c[q] - m;
                            double dd = ce[q] + me + U32 * (fabs(dq) + ce[q] + me);
                            v += dq * dq / 4.0;
                            ve += dd * (2.0 * fabs(dq) + dd) / 4.0;
                        }
                        ve += gamma_n(5) * (v + ve);
                        pv[p] = v;
                        pve[p] = 2.0 * ve; /* FMA contraction slack */
                    }
            }
            /* 3. band value, split/keep decisions and Eq. 2's active mask; parents
             *    (depth d-1) are decided before their children (depth d). */
            for (int d = 0; d <= D; d++) {
                int64_t n = side_len(d);
                for (int64_t i = 0; i < n; i++)
                    for (int64_t j = 0; j < n; j++) {
                        int64_t p = level_offset(d) + morton(i, j);
                        double nb[4], nbe[4];
                        int64_t ni[4] = {i - 1, i + 1, i, i};
                        int64_t nj[4] = {j, j, j - 1, j + 1};
                        for (int q = 0; q < 4; q++) {
                            if (ni[q] >= 0 && ni[q] < n && nj[q] >= 0 && nj[q] < n) {
                                int64_t pq = level_offset(d) + morton(ni[q], nj[q]);
                                nb[q] = pw[pq]; nbe[q] = pe[pq];
                            } else {
                                int sd = ni[q] < 0 ? 0 : ni[q] >= n ? 1 : nj[q] < 0 ? 2 : 3;
                                int64_t t = sd < 2 ? nj[q] : ni[q];
                                int64_t h = halo_offset(d) + sd * n + t;
                                nb[q] = ph[h]; nbe[q] = phe[h];
                            }
                        }
                        /* ES-HyperNEAT band: max(min(d_top, d_bottom), min(d_left, d_right)) */
                        double dl = fabs(pw[p] - nb[0]), dr = fabs(pw[p] - nb[1]);
                        double db = fabs(pw[p] - nb[2]), dt = fabs(pw[p] - nb[3]);
                        double B = fmax(fmin(dt, db), fmin(dl, dr));
                        double Be = 0.0, dmax = fmax(fmax(dl, dr), fmax(db, dt));
                        for (int q = 0; q < 4; q++) Be = fmax(Be, pe[p] + nbe[q]);
                        Be += 2.0 * U32 * dmax;
                        /* fp64 decisions */
                        int sp64 = d < D && pv[p] > theta;
                        int ke64 = !sp64 && B > band && (w_min <= 0.0 || fabs(pw[p]) > w_min);
                        int ac64 = 1;
                        /* the same decisions with their fp32 margins (0 / 1 / 2 = uncertain) */
                        int sp3 = d == D ? 0 : decide_gt(pv[p], theta, TIE_MARGIN + pve[p]);
                        int bp3 = decide_gt(B, band, TIE_MARGIN + Be);
                        int wp3 = w_min > 0.0 ? decide_gt(fabs(pw[p]), w_min, TIE_MARGIN + pe[p]) : 1;
                        int ke3 = and3(and3(not3(sp3), bp3), wp3);
                        int ac3 = 1;
                        if (d > 0) {
                            int64_t par = level_offset(d - 1) + morton(i >> 1, j >> 1);
                            ac64 = act64[par] && pv[par] > theta;
                            ac3 = and3(act3[par], decide_gt(pv[par], theta, TIE_MARGIN + pve[par]));
                        }
                        act64[p] = (uint8_t)ac64;
                        act3[p] = (uint8_t)ac3;
                        int kg64 = ke64 && ac64;
                        int kg3 = and3(ke3, ac3);
                        int64_t o = r * NT + p;
                        if (bnd) bnd[o] = B;
                        if (bnd_err) bnd_err[o] = Be;
                        if (keep_eager) keep_eager[o] = (uint8_t)ke64;
                        if (unc_eager) unc_eager[o] = (uint8_t)(ke3 == 2);
                        if (keep_gated) keep_gated[o] = (uint8_t)kg64;
                        if (unc_gated) unc_gated[o] = (uint8_t)(kg3 == 2);
                        if (split) split[o] = (uint8_t)sp64;
                    }
            }
            for (int64_t p = 0; p < NT; p++) {
                int64_t o = r * NT + p;
                if (w) w[o] = pw[p];
                if (w_err) w_err[o] = pe[p];
                if (var) var[o] = pv[p];
                if (var_err) var_err[o] = pve[p];
            }
            for (int64_t h = 0; h < NH; h++) {
                if (w_halo) w_halo[r * NH + h] = ph[h];
                if (halo_err) halo_err[r * NH + h] = phe[h];
            }
        }
        free(pw); free(pe); free(ph); free(phe); free(pv); free(pve); free(act64); free(act3); free(val); free(er);
    }
    for (int k = 0; k < G; k++) genome_free(&gen[k]);
    free(gen);
    return ORA_OK;
}

/* ---- lazy ES-HyperNEAT quadtree (Fig. 1, left; Section 2) ----------------- */

typedef struct {
    const genome_t *G;
    int side, D;
    double a, b, theta, band, w_min;
    uint8_t *keep;
    double *val, *er;
    int64_t evals;
} lazy_t;

static double lazy_w(lazy_t *c, double x, double y)
{
    double in[5], e;
    query_inputs(c->side, c->a, c->b, x, y, in);
    c->evals++;
    return cppn_eval(c->G, in, c->val, c->er, &e);
}

/* variance of the four children of cell (d, i, j), evaluated on demand */
static double lazy_var(lazy_t *c, int d, int64_t i, int64_t j)
{
    double v[4], m = 0.0, s = 0.0;
    for (int q = 0; q < 4; q++) {
        v[q] = lazy_w(c, coord(d + 1, 2 * i + (q & 1)), coord(d + 1, 2 * j + (q >> 1)));
        m += v[q] / 4.0;
    }
    for (int q = 0; q < 4; q++) s += (v[q] - m) * (v[q] - m) / 4.0;
    return s;
}

/* Visit a cell whose four children lie at depth d; (pi, pj) is the cell at
 * depth d-1 (the root when d == 0). A child is subdivided when its variance
 * exceeds theta and it is above the maximum depth; otherwise it is a leaf and
 * is kept when its band value, taken from CPPN queries at distance 2^-d left,
 * right, below and above it, exceeds the band threshold. */
static void lazy_visit(lazy_t *c, int d, int64_t pi, int64_t pj)
{
    for (int q = 0; q < 4; q++) {
        int64_t i = 2 * pi + (q & 1), j = 2 * pj + (q >> 1);
        if (d < c->D && lazy_var(c, d, i, j) > c->theta) {
            lazy_visit(c, d + 1, i, j);
            continue;
        }
        double x = coord(d, i), y = coord(d, j), s = 1.0 / (double)((int64_t)1 << d);
        double w = lazy_w(c, x, y);
        double dl = fabs(w - lazy_w(c, x - s, y)), dr = fabs(w - lazy_w(c, x + s, y));
        double db = fabs(w - lazy_w(c, x, y - s)), dt = fabs(w - lazy_w(c, x, y + s));
        if (fmax(fmin(dt, db), fmin(dl, dr)) > c->band && (c->w_min <= 0.0 || fabs(w) > c->w_min))
            c->keep[level_offset(d) + morton(i, j)] = 1;
    }
}

/* Lazy discovery for genomes [g0, g1) and S slots (same source conventions as
 * ora_discover). keep[r * N_total + global index] = 1 for each kept position;
 * evals[r] (optional) = CPPN queries the lazy tree issued. */
int ora_lazy(const int64_t *node_ptr, const int32_t *node_id, const int32_t *node_kind,
             const int32_t *node_act, const float *node_bias, const int64_t *conn_ptr,
             const int32_t *conn_src, const int32_t *conn_dst, const float *conn_w, const uint8_t *conn_en,
             int g0, int g1, int S, const float *src_a, const float *src_b, const int32_t *src_side,
             int per_genome, const int32_t *src_count, int D, double theta, double band, double w_min,
             uint8_t *keep, int64_t *evals, int nthreads)
{
    if (D < 0 || D > MAX_DEPTH || g1 < g0 || S < 0) return ORA_ERR_ARG;
    int G = g1 - g0;
    const int64_t NT = level_offset(D + 1);
    genome_t *gen = calloc(G > 0 ? G : 1, sizeof(genome_t));
    if (!gen) return ORA_ERR_ALLOC;
    int rc = ORA_OK;
    for (int k = 0; k < G && rc == ORA_OK; k++)
        rc = genome_build(&gen[k], g0 + k, node_ptr, node_id, node_kind, node_act, node_bias, conn_ptr,
                          conn_src, conn_dst, conn_w, conn_en);
    if (rc != ORA_OK) {
        for (int k = 0; k < G; k++) genome_free(&gen[k]);
        free(gen);
        return rc;
    }
    int64_t pairs = (int64_t)G * S;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t r = 0; r < pairs; r++) {
        int gl = (int)(r / S), s = (int)(r % S), g = g0 + gl;
        memset(keep + r * NT, 0, (size_t)NT);
        if (evals) evals[r] = 0;
        if (per_genome && src_count && s >= src_count[g]) continue;
        int64_t si = per_genome ? (int64_t)g * S + s : s;
        lazy_t c;
        c.G = &gen[gl];
        c.side = src_side[si];
        c.a = (double)src_a[si];
        c.b = (double)src_b[si];
        c.D = D; c.theta = theta; c.band = band; c.w_min = w_min;
        c.keep = keep + r * NT;
        c.val = malloc(sizeof(double) * gen[gl].n);
        c.er = malloc(sizeof(double) * gen[gl].n);
        c.evals = 0;
        lazy_visit(&c, 0, 0, 0);
        if (evals) evals[r] = c.evals;
        free(c.val); free(c.er);
    }
    for (int k = 0; k < G; k++) genome_free(&gen[k]);
    free(gen);
    return ORA_OK;
}

/* ---- decisions at individual positions, by definition -------------------- */

/* For genome g and one query slot (a, b, side): at each listed grid position
 * (d[k], i[k], j[k]) of a depth-D grid, the CPPN output, its V, B, the eager
 * keep decision in fp64 and whether it is uncertain at the fp32 margins, all
 * from direct CPPN queries (children, neighbours). For sampled checks of grids
 * too large to evaluate whole. */
int ora_keep_at(int g, const int64_t *node_ptr, const int32_t *node_id, const int32_t *node_kind,
                const int32_t *node_act, const float *node_bias, const int64_t *conn_ptr, const int32_t *conn_src,
                const int32_t *conn_dst, const float *conn_w, const uint8_t *conn_en, float src_a, float src_b,
                int side, int D, double theta, double band, double w_min, int64_t n, const int32_t *dd,
                const int64_t *ii, const int64_t *jj, double *w_out, double *w_err, double *var_out, double *bnd_out,
                uint8_t *keep, uint8_t *unc, int nthreads)
{
    genome_t G;
    int rc = genome_build(&G, g, node_ptr, node_id, node_kind, node_act, node_bias, conn_ptr, conn_src, conn_dst,
                          conn_w, conn_en);
    if (rc != ORA_OK) return rc;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel
#endif
    {
        double *val = malloc(sizeof(double) * G.n), *er = malloc(sizeof(double) * G.n);
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 64)
#endif
        for (int64_t k = 0; k < n; k++) {
            const int d = dd[k];
            const int64_t i = ii[k], j = jj[k];
            double in[5], e, we;
            query_inputs(side, src_a, src_b, coord(d, i), coord(d, j), in);
            const double w = cppn_eval(&G, in, val, er, &we);
            /* variance of the four children and its bound (as ora_discover) */
            double V = 0.0, Ve = 0.0;
            if (d < D) {
                double c[4], ce[4], m = 0.0, me = 0.0, cm = 0.0;
                for (int q = 0; q < 4; q++) {
                    query_inputs(side, src_a, src_b, coord(d + 1, 2 * i + (q & 1)), coord(d + 1, 2 * j + (q >> 1)), in);
                    c[q] = cppn_eval(&G, in, val, er, &ce[q]);
                    m += c[q] / 4.0; me += ce[q] / 4.0; cm += fabs(c[q]) / 4.0;
                }
                me += gamma_n(4) * cm;
                for (int q = 0; q < 4; q++) {
                    double dq = c[q] - m, dl = ce[q] + me + U32 * (fabs(dq) + ce[q] + me);
                    V += dq * dq / 4.0;
                    Ve += dl * (2.0 * fabs(dq) + dl) / 4.0;
                }
                Ve += gamma_n(5) * (V + Ve);
                Ve *= 2.0;
            }
            /* band value from the four neighbours at distance 2^-d */
            const int64_t ni[4] = {i - 1, i + 1, i, i}, nj[4] = {j, j, j - 1, j + 1};
            double nb[4], nbe[4];
            for (int q = 0; q < 4; q++) {
                query_inputs(side, src_a, src_b, coord(d, ni[q]), coord(d, nj[q]), in);
                nb[q] = cppn_eval(&G, in, val, er, &nbe[q]);
            }
            double dl = fabs(w - nb[0]), dr = fabs(w - nb[1]), db = fabs(w - nb[2]), dt = fabs(w - nb[3]);
            double B = fmax(fmin(dt, db), fmin(dl, dr)), Be = 0.0, dmax = fmax(fmax(dl, dr), fmax(db, dt));
            for (int q = 0; q < 4; q++) Be = fmax(Be, we + nbe[q]);
            Be += 2.0 * U32 * dmax;
            int sp64 = d < D && V > theta;
            int sp3 = d == D ? 0 : decide_gt(V, theta, TIE_MARGIN + Ve);
            int bp3 = decide_gt(B, band, TIE_MARGIN + Be);
            int wp3 = w_min > 0.0 ? decide_gt(fabs(w), w_min, TIE_MARGIN + we) : 1;
            int k3 = and3(and3(not3(sp3), bp3), wp3);
            if (w_out) w_out[k] = w;
            if (w_err) w_err[k] = we;
            if (var_out) var_out[k] = V;
            if (bnd_out) bnd_out[k] = B;
            keep[k] = (uint8_t)(!sp64 && B > band && (w_min <= 0.0 || fabs(w) > w_min));
            unc[k] = (uint8_t)(k3 == 2);
            (void)e;
        }
        free(val); free(er);
    }
    genome_free(&G);
    return ORA_OK;
}

/*
 * Connection types (Section 6, its connection-type taxonomy): a connection from
 * source s to target t is a self-loop when s = t, and otherwise forward when
 * y_s < y_t, backward when y_s > y_t and lateral when y_s = y_t. For a query
 * slot at (a, b): on the outgoing side the slot is the source and the grid
 * position the target; on the incoming side the position is the source and
 * the slot the target. Codes: 0 forward, 1 backward, 2 lateral, 3 self.
 * Coordinates are exact dyadic rationals, so the comparisons are exact.
 */
int ora_conn_type(double a, double b, int side, int d, int64_t i, int64_t j)
{
    double x = coord(d, i), y = coord(d, j);
    double xs = side == 0 ? a : x, ys = side == 0 ? b : y;   /* source */
    double xt = side == 0 ? x : a, yt = side == 0 ? y : b;   /* target */
    if (xs == xt && ys == yt) return 3;
    if (ys < yt) return 0;
    if (ys > yt) return 1;
    return 2;
}

/* ora_conn_type at n positions given by global index. */
int ora_conn_types(double a, double b, int side, int64_t n, const int64_t *gidx, uint8_t *type)
{
    if (n < 0 || (n > 0 && (!gidx || !type))) return ORA_ERR_ARG;
    for (int64_t k = 0; k < n; k++) {
        int d = 0;
        while (level_offset(d + 1) <= gidx[k]) d++;
        int64_t m = gidx[k] - level_offset(d), i = 0, j = 0;
        for (int bit = 0; bit < 31; bit++) {           /* Morton decode */
            i |= ((m >> (2 * bit)) & 1) << bit;
            j |= ((m >> (2 * bit + 1)) & 1) << bit;
        }
        type[k] = (uint8_t)ora_conn_type(a, b, side, d, i, j);
    }
    return ORA_OK;
}
