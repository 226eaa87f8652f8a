/*
 * emr.h: C ABI of libemr, a GB300 (sm_103a) implementation of the eager
 * multi-resolution substrate-discovery hot path of EMR-HyperNEAT
 * ("Tensor-Accelerated Eager Multi-Resolution Grids for Evolving Large-Scale
 * Substrates", GECCO Companion '26).
 *
 * The method (Section 3): precompute the multi-resolution grid of Eq. 1,
 * query every genome's CPPN at every grid position (W = vmap(CPPN)(s, T)),
 * compute each cell's variance bottom-up from its four children, and filter
 * with the division threshold (Eq. 2) and ES-HyperNEAT's band threshold; the
 * surviving positions become each genome's connection list.
 *
 * Conventions shared by every call
 * --------------------------------
 * Grid (Eq. 1): depth d in [0, D] holds the 4^{d+1} points
 *   x = (2i+1)/2^{d+1} - 1, y = (2j+1)/2^{d+1} - 1, i, j in [0, 2^{d+1}).
 * Position numbering: global index = level_off[d] + m, level_off[d] =
 *   (4^{d+1} - 4)/3, m = Morton code of (i, j) (bit k of i -> bit 2k, bit k of
 *   j -> bit 2k+1). The children of m at depth d are 4m + a + 2b at depth
 *   d+1 for child (2i+a, 2j+b). N_total = (4^{D+2} - 4)/3.
 * Halo: the band test of a depth-d point looks at its 4 neighbours at
 *   distance 2^-d; those outside [-1,1]^2 are the halo points, numbered
 *   halo_off[d] + side * 2^{d+1} + t, halo_off[d] = 8 (2^d - 1);
 *   side 0: (i = -1, j = t), 1: (i = 2^{d+1}, j = t), 2: (i = t, j = -1),
 *   3: (i = t, j = 2^{d+1}). N_halo = 8 (2^{D+1} - 1).
 * Bit planes: one bit per position, levels padded to whole 32-bit words
 *   (device uint32 [pair][n_words], 16-byte aligned). mask and split are
 *   position-major: position (d, m) is bit (m % 32) of word word_off[d] + m / 32;
 *   bits past a level's 4^{d+1} positions (depths 0 and 1) are 0. band_bits
 *   is position-major at depths 0..2 and quad-major from depth 3: position
 *   (d, m) is bit (m / 4) % 32 of word word_off[d] + 4 (m / 128) + m % 4 (the
 *   four words of each 128-position block hold children 0..3 of its 32 quads).
 * Query slots: a (genome, slot) pair ("pair") evaluates CPPN(a, b, x, y, 1)
 *   for an outgoing slot (source node at (a, b)) or CPPN(x, y, a, b, 1) for an
 *   incoming slot (target node at (a, b)) over every grid position; the CPPN
 *   input order (x1, y1, x2, y2) is the paper's (Section 2), the fifth input
 *   is the bias, fixed at 1. Pair r = g * S + s.
 * Filter (Section 3.2, Eq. 2, Theorem 1): V(p) = population variance of the
 *   CPPN outputs at p's four children (0 at depth D); split(p) = d < D and
 *   V(p) > theta; B(p) = max(min(|w_p - w_up|, |w_p - w_down|),
 *   min(|w_p - w_left|, |w_p - w_right|)) (ES-HyperNEAT's band value);
 *   keep_eager(p) = !split(p) and B(p) > band and (w_min <= 0 or |w_p| > w_min);
 *   keep_gated(p) = keep_eager(p) and active(p), active per Eq. 2.
 *
 * Memory and streams: the caller owns every buffer. Device pointers must be
 * device memory of the current CUDA device; host pointers are plain host
 * memory unless a call says "pinned". Calls that take a stream are
 * asynchronous on it unless stated; errors are returned as status codes and
 * never thrown; on error no kernel has been launched unless stated.
 */
#ifndef EMR_H
#define EMR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int emr_status;
#define EMR_OK 0
#define EMR_ERR_ARG 1      /* bad argument (null pointer, size, enum, malformed genome) */
#define EMR_ERR_CYCLE 2    /* a genome's enabled connections contain a cycle */
#define EMR_ERR_RANGE 3    /* a size beyond a documented limit (depth, nodes, edges) */
#define EMR_ERR_CAPACITY 4 /* an output buffer is too small; true sizes are reported */
#define EMR_ERR_CUDA 5     /* a CUDA runtime call or launch failed */
#define EMR_ERR_TIMEOUT 6  /* a host-side wait gave up */
#define EMR_ERR_ALLOC 7    /* host allocation failed */

#define EMR_MAX_DEPTH 14   /* global indices fit int32 up to depth 14 (N_total(14) = 1.43e9) */
#define EMR_MAX_VARYING 64 /* per genome and query side: CPPN nodes whose value varies over the grid */
#define EMR_MAX_VEDGES 512 /* per genome: connections between such nodes */

enum { EMR_ACT_IDENTITY = 0, EMR_ACT_SIGMOID = 1, EMR_ACT_TANH = 2, EMR_ACT_GAUSS = 3,
       EMR_ACT_SIN = 4, EMR_ACT_ABS = 5 };
enum { EMR_KIND_X1 = 0, EMR_KIND_Y1 = 1, EMR_KIND_X2 = 2, EMR_KIND_Y2 = 3, EMR_KIND_BIAS = 4,
       EMR_KIND_HIDDEN = 5, EMR_KIND_OUTPUT = 6 };
enum { EMR_SIDE_OUT = 0, EMR_SIDE_IN = 1 };
enum { EMR_EAGER = 0, EMR_GATED = 1 };
/* Connection types (Section 6, connection type taxonomy), as bits of a filter
 * and, in emr_conn_types, as codes 0..3 in this order: forward (source below
 * target, y_s < y_t), backward (y_s > y_t), lateral (y_s = y_t), self-loop (s = t). */
enum { EMR_CONN_F = 1, EMR_CONN_B = 2, EMR_CONN_L = 4, EMR_CONN_S = 8, EMR_CONN_ALL = 15 };
/* The six substrate configurations of Section 6 (its table), see emr_substrate_config. */
enum { EMR_SUBSTRATE_FEEDFORWARD = 0, EMR_SUBSTRATE_HH = 1, EMR_SUBSTRATE_BACKWARD = 2,
       EMR_SUBSTRATE_LATERAL = 3, EMR_SUBSTRATE_SELF = 4, EMR_SUBSTRATE_FULL = 5 };

/* Grid descriptor (Eq. 1): sizes and offsets only, no positions are stored;
 * kernels generate coordinates from (depth, Morton index). */
typedef struct {
    int32_t D;
    int32_t reserved;
    int64_t n_total;                      /* (4^{D+2} - 4) / 3 positions */
    int64_t n_halo;                       /* 8 (2^{D+1} - 1) halo points */
    int64_t n_words;                      /* bit-plane words per pair */
    int64_t chunk;                        /* streaming chunk in positions (0 = none) */
    int64_t level_off[EMR_MAX_DEPTH + 2]; /* [d] first global index of depth d; [D+1] = n_total */
    int64_t halo_off[EMR_MAX_DEPTH + 2];  /* [d] first halo index of depth d; [D+1] = n_halo */
    int64_t word_off[EMR_MAX_DEPTH + 2];  /* [d] first bit-plane word of depth d; [D+1] = n_words */
} emr_grid;                               /* offset entries past D + 1 repeat the [D + 1] totals */

/* Query slots. Shared by all genomes (per_genome = 0: arrays of S) or one
 * list per genome (per_genome = 1: arrays of P * S, row g). count (per-genome
 * mode, optional) gives the number of valid slots of each genome; slots past
 * it evaluate to the constant 0 and keep nothing. Host and device copies hold
 * the same values: the host copy schedules work, the device copy is read by
 * kernels. */
typedef struct {
    int32_t S;
    int32_t per_genome;
    const float *a_host, *b_host;      /* node coordinates */
    const int32_t *side_host;          /* EMR_SIDE_OUT / EMR_SIDE_IN */
    const int32_t *count_host;         /* optional, [P] */
    const float *a_dev, *b_dev;
    const int32_t *side_dev;
    const int32_t *count_dev;          /* optional, [P] */
} emr_query;

/* ---- a1: grid descriptor ------------------------------------------------ */

/* Fill *grid for maximum depth D (Eq. 1, Section 3.1; Table 1 "grid
 * construction"). chunk: positions per streaming chunk for emr_stream (0 =
 * no chunking; otherwise a power of two >= 4096). Host only, no allocation.
 * Errors: EMR_ERR_ARG (null grid, bad chunk), EMR_ERR_RANGE (D outside [0, 14]). */
emr_status emr_grid_build(int32_t D, int64_t chunk, emr_grid *grid);

/* Depth d and grid indices (i, j) of global index gidx (inverse of the
 * numbering above). Returns EMR_ERR_RANGE when gidx is negative or past
 * depth EMR_MAX_DEPTH. */
emr_status emr_index_to_ij(int64_t gidx, int32_t *d, int32_t *i, int32_t *j);

/* ---- a2: population packing (host) -------------------------------------- */

/* Bytes emr_pack_population writes for this population: each genome's records
 * take the room of its input nodes and connections, so that genomes pack
 * independently (on several host threads) straight into the blob. */
emr_status emr_pack_size(int32_t P, const int64_t *node_ptr, const int64_t *conn_ptr, size_t *bytes);

/* Pack P NEAT genomes (Section 2; the TensorNEAT genomes of Section 5.1) into
 * one position-independent blob. Genome g owns nodes [node_ptr[g],
 * node_ptr[g+1]) and connections [conn_ptr[g], conn_ptr[g+1]). Nodes: unique
 * id, kind (EMR_KIND_*), activation (EMR_ACT_*, hidden and output only) and
 * bias; exactly one output per genome. Connections: (source id, destination
 * id, weight, enabled); disabled connections are ignored. A node's value is
 * act(bias + sum of weight * source value over its enabled in-connections).
 *
 * The packer orders each genome topologically (Kahn's algorithm, ties by node
 * id), merges parallel connections (same source and destination) into one
 * whose weight is their fp32 sum in connection order, drops connections whose
 * weight is then 0 (they add 0 for any finite source value), drops nodes that
 * cannot reach the output, folds input connections into per-node input weights
 * and records, per query side, which grid coordinates (x, y or both) each node
 * depends on. The blob is plain bytes: copy it to device memory unchanged (any
 * 16-byte aligned address) and pass both copies to the eval calls.
 * Errors: EMR_ERR_ARG (null pointer, malformed genome: unknown id, duplicate
 * id, not exactly one output, connection into an input), EMR_ERR_CYCLE,
 * EMR_ERR_RANGE (more than EMR_MAX_VARYING varying nodes or EMR_MAX_VEDGES
 * edges between them), EMR_ERR_CAPACITY (cap too small; *used = bytes needed).
 * *bad_genome (optional) receives the index of the offending genome or -1. */
emr_status emr_pack_population(int32_t P, const int64_t *node_ptr, const int32_t *node_id,
                               const int32_t *node_kind, const int32_t *node_act, const float *node_bias,
                               const int64_t *conn_ptr, const int32_t *conn_src, const int32_t *conn_dst,
                               const float *conn_w, const uint8_t *conn_enabled, void *buf, size_t cap,
                               size_t *used, int32_t *bad_genome);

/* Genome ranges. The packer reads genome g through node_ptr[g] and conn_ptr[g]
 * as absolute offsets into the node and connection arrays, so genomes
 * [g0, g1) of a population are packed on their own by passing P = g1 - g0,
 * node_ptr + g0 and conn_ptr + g0 (the other arrays unchanged): the blob then
 * holds those genomes as genomes 0 .. g1 - g0 - 1. With per-genome query slots,
 * the query of such a range is rows g0 .. g1 - 1 of the slot arrays. */

/* Population-parallel split (Section 3, Table 1: the CPPN query, variance and
 * mask stages are O(4^D / P) work over the population): n_parts contiguous
 * genome ranges of balanced estimated cost for this pack and query. A pair's
 * cost is the packer's per-query work estimate of its genome on the slot's
 * query side plus the filter's per-query work; constant-output pairs and unused
 * per-genome slots count 1. Writes g_begin[0 .. n_parts] (host int32):
 * part k is genomes [g_begin[k], g_begin[k+1]), g_begin[0] = 0,
 * g_begin[n_parts] = P, non-decreasing (a part may be empty when n_parts > P).
 * Concatenating the parts' connection lists in part order gives the lists of
 * the whole population (pair r = g * S + s). Host only.
 * Errors: EMR_ERR_ARG (null pointer, n_parts <= 0, bad side, not a pack). */
emr_status emr_partition_genomes(const void *pack_host, const emr_query *q, int32_t n_parts, int32_t *g_begin);

/* The packer's state kept between calls: up to 15 host worker threads (started
 * on first use; starting them costs as much as packing a few dozen genomes;
 * after a call they watch for the next one for 0.4 ms before they sleep) and
 * its per-thread scratch (grown to the largest genome packed). This
 * is libemr's one process-wide state besides emr_eval_filter_noalloc's static
 * device array; it holds no results, only scratch. emr_pack_release joins the
 * worker threads and frees the buffers; the next emr_pack_population (or
 * emr_assemble, which shares the workers) recreates them. Libemr also joins
 * the workers when it is unloaded or the process exits. Must not be called
 * while another thread is inside emr_pack_population or emr_assemble. */
void emr_pack_release(void);

/* Summary of a packed blob: population size and, per query side, the largest
 * number of varying nodes. Any output pointer may be NULL. */
emr_status emr_pack_info(const void *pack_host, int32_t *P, int32_t *max_varying_out,
                         int32_t *max_varying_in);

/* ---- device workspace and per-pair specialisation ------------------------- */

/* Bytes of device workspace the eval calls need for this pack and query
 * (per-pair specialised CPPN records, scratch and the pair schedule). */
emr_status emr_eval_workspace_size(const void *pack_host, const emr_query *q, size_t *bytes);

/* Specialise every (genome, slot) pair into ws (Section 3.1: W = CPPN(s, T)
 * with the slot's node s fixed): the slot's node coordinates and the bias are
 * folded with every CPPN node that does not vary over the grid into per-node
 * constants, and the pairs are ordered by estimated cost, heaviest first.
 * pack_dev: device copy of the blob from emr_pack_population; q: host and
 * device copies of the slots. Must precede emr_eval / emr_eval_filter with the
 * same pack and query (stream order). Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY
 * (ws_bytes too small), EMR_ERR_CUDA. */
emr_status emr_eval_prepare(const void *pack_host, const void *pack_dev, const emr_query *q, void *ws,
                            size_t ws_bytes, void *stream);

/* ---- a3: batched CPPN evaluation ---------------------------------------- */

/* W = CPPN(s, T) at every grid position (Section 3.1, Eq. 1; Table 1 "CPPN
 * query"), materialised. out: device float [P * S][n_total] (pair-major,
 * global index; 16-byte aligned); out_halo: device float [P * S][n_halo] or
 * NULL (then halo points are not evaluated). ws: prepared by
 * emr_eval_prepare. Each position is evaluated once; coordinates are
 * generated in the kernel. Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY, EMR_ERR_RANGE
 * (more than 2^31 - 1 tiles: use emr_stream), EMR_ERR_CUDA. */
emr_status emr_eval(const void *pack_host, const emr_query *q, const emr_grid *grid, float *out, float *out_halo,
                    void *ws, size_t ws_bytes, void *stream);

/* Chunks of a grid (the chunking emr_stream uses; Section 5.2 and Section 6
 * stream depths 8..13 because W no longer fits): grid->chunk positions per
 * chunk in whole 64 x 64 tiles (0 = one chunk), the tile of depths 0..4 in the
 * lowest chunk, chunks numbered 0 .. *n_chunks - 1 in ascending global index.
 * Chunk chunk_idx covers global indices [*pos_beg, *pos_end). n_chunks, pos_beg,
 * pos_end may each be NULL (with both position pointers NULL only *n_chunks is
 * written and chunk_idx is not checked). Host only. Errors: EMR_ERR_ARG (bad
 * grid, chunk not a multiple of 4096), EMR_ERR_RANGE (chunk_idx outside). */
emr_status emr_grid_chunk(const emr_grid *grid, int64_t chunk_idx, int64_t *n_chunks, int64_t *pos_beg,
                          int64_t *pos_end);

/* emr_eval over one chunk of the grid (emr_grid_chunk), for materialising W one
 * chunk at a time when the whole grid does not fit (Section 5.2: the paper
 * streams W through host memory at depth 7 and beyond). out: device float
 * [P * S][pos_end - pos_beg], pair r's output at global index g in
 * out[r][g - pos_beg] (16-byte aligned); out_halo: NULL or the whole-grid halo
 * buffer of emr_eval (only the halo points next to the chunk's tiles are
 * written). ws: prepared by emr_eval_prepare. Every chunk's values equal
 * emr_eval's at the same positions. Errors: EMR_ERR_ARG, EMR_ERR_RANGE
 * (chunk_idx outside), EMR_ERR_CAPACITY, EMR_ERR_CUDA. */
emr_status emr_eval_chunk(const void *pack_host, const emr_query *q, const emr_grid *grid, int64_t chunk_idx,
                          float *out, float *out_halo, void *ws, size_t ws_bytes, void *stream);

/* ---- a4, a5: variance and band/threshold filter --------------------------- */

/* Filter a materialised evaluation (Section 3.2, Eq. 2; Theorem 1's band
 * threshold). out/out_halo as written by emr_eval. Writes three bit planes,
 * device uint32 [P * S][n_words] each: split (d < D and V > theta), band_bits
 * (B > band and the weight filter) and mask (emr_mask_combine of the two in
 * the given mode); var_dbg (optional, device float [P * S][n_total]) receives
 * V(p). theta >= 0, band >= 0, w_min >= 0 (0 = weight filter off).
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_variance_filter(const float *out, const float *out_halo, const emr_grid *grid, int32_t P,
                               int32_t S, float theta, float band, float w_min, int32_t mode, uint32_t *mask,
                               uint32_t *split, uint32_t *band_bits, float *var_dbg, void *stream);

/* Keep mask from the two planes: mask = band_bits AND NOT split (a depth-D
 * position never splits), and for EMR_GATED also AND active (Eq. 2: every
 * ancestor split). Bits past a level's positions are cleared.
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_mask_combine(const uint32_t *split, const uint32_t *band_bits, const emr_grid *grid,
                            int32_t n_pairs, int32_t mode, uint32_t *mask, void *stream);

/* emr_mask_combine, then keep only connections whose type (Section 6
 * taxonomy) is in types (EMR_CONN_* bits; EMR_CONN_ALL keeps every type). A
 * connection joins pair r's query slot (q's slot r mod S, or row r in
 * per-genome mode) and a grid position: on the outgoing side the slot is the
 * source, on the incoming side the target. n_pairs must be a multiple of q->S.
 * The comparisons are exact: grid coordinates are dyadic and computed exactly
 * in fp32, and the slot coordinates are the fp32 values of q.
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_mask_combine_types(const uint32_t *split, const uint32_t *band_bits, const emr_query *q,
                                  const emr_grid *grid, int32_t n_pairs, int32_t mode, int32_t types,
                                  uint32_t *mask, void *stream);

/* Connection types enabled by one of the six substrate configurations of
 * Section 6 (EMR_SUBSTRATE_*), and whether it runs hidden-to-hidden rounds
 * (*hidden_rounds = 1; 0 for the feedforward configuration, which skips the
 * second phase): feedforward F; hidden-to-hidden F (+ rounds); backward F, B;
 * lateral F, L; self F, S; full recurrent F, B, L, S. Either output may be
 * NULL. Host only. Errors: EMR_ERR_ARG (unknown config). */
emr_status emr_substrate_config(int32_t config, int32_t *types, int32_t *hidden_rounds);

/* ---- a3+a4+a5 fused ------------------------------------------------------ */

/* Evaluate and filter in one kernel, without materialising the CPPN outputs:
 * each tile of positions evaluates its points and the ring of neighbours it
 * needs, takes each parent cell's variance from its four children in registers
 * and each position's band value from shared memory, and writes only the split
 * and band_bits planes (as emr_variance_filter) plus, when out is not NULL, the
 * CPPN output at positions whose band test passed (other entries of out are
 * left untouched). Follow with emr_mask_combine. ws: prepared by
 * emr_eval_prepare. Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY, EMR_ERR_RANGE,
 * EMR_ERR_CUDA. */
emr_status emr_eval_filter(const void *pack_host, const emr_query *q, const emr_grid *grid, float theta,
                           float band, float w_min, uint32_t *split, uint32_t *band_bits, float *out, void *ws,
                           size_t ws_bytes, void *stream);

/* ---- a7: chunked streaming --------------------------------------------------- */

/* Bytes of device workspace emr_stream needs: the per-pair records, the
 * resident split plane (n_pairs x n_words x 4 bytes) and two chunk buffers
 * (band bits, mask, compaction workspace and chunk_cap list entries each; the
 * kept weights are recomputed from the records, so no outputs are stored). */
emr_status emr_stream_workspace_size(const void *pack_host, const emr_query *q, const emr_grid *grid,
                                     int64_t chunk_cap, size_t *bytes);

/* The whole eager path (emr_eval_prepare, emr_eval_filter, emr_mask_combine
 * with EMR_EAGER, emr_compact) over grids too large to hold, in chunks of
 * grid->chunk positions (whole 64 x 64 tiles; 0 = one chunk), with only the
 * compacted lists leaving the GPU (Section 5.2 and Section 6 stream depths
 * 8..13 through host memory or disk; here only the kept int32 indices and fp32
 * weights are copied out). Chunks run from the highest global index down, so
 * each chunk's split bits (written by its children) are final when it is
 * filtered; two chunk buffers alternate on `stream` while a second,
 * library-created stream copies the previous chunk's lists to the host.
 *
 * h_idx, h_w: host arrays of cap entries (pinned memory keeps the copies
 * asynchronous); on return pair r's list is [offsets[r], offsets[r+1]) in
 * ascending global index, counts[r] its length (host int64 [n_pairs], offsets
 * [n_pairs + 1]). chunk_cap: list entries one chunk may produce (device
 * buffers). Synchronous: returns when the lists are on the host.
 * This is emr_stream_mode with EMR_EAGER and EMR_CONN_ALL.
 * Errors: EMR_ERR_ARG; EMR_ERR_CAPACITY (ws too small, or a chunk or the total
 * exceeded chunk_cap / cap: counts hold the true totals, the lists are
 * incomplete); EMR_ERR_TIMEOUT when a host wait exceeds timeout_ms (0 = no
 * limit): queued work is still running then and writes into ws and the host
 * arrays, so synchronise the device before reusing them; EMR_ERR_CUDA.
 * Allocates per call a copy stream, four events and 16 (n_pairs + 1) bytes of
 * pinned host staging. On EMR_ERR_TIMEOUT the pinned staging is not freed
 * (copies still queued may write into it, and freeing pinned memory would wait
 * for them): each timed-out call leaks those 16 (n_pairs + 1) bytes of pinned
 * host memory until the process exits; the stream and events are released. */
emr_status emr_stream(const void *pack_host, const void *pack_dev, const emr_query *q, const emr_grid *grid,
                      float theta, float band, float w_min, void *ws, size_t ws_bytes, int64_t chunk_cap,
                      int32_t *h_idx, float *h_w, int64_t cap, int64_t *counts, int64_t *offsets,
                      int64_t timeout_ms, void *stream);

/* emr_stream with a mode and a connection-type filter (types as in
 * emr_mask_combine_types, applied per chunk when its mask is formed). GATED
 * (Eq. 2) needs every ancestor's split bit, which the descending stream has
 * only at its end: the eager lists (a superset) are collected as in
 * emr_stream, then each entry is checked against the resident split plane on
 * the device (entries copied back chunk_cap at a time) and the lists are
 * compacted in place on the host. cap must hold the eager lists; on
 * EMR_ERR_CAPACITY counts hold the eager totals and no gate is applied.
 * Errors as emr_stream. */
emr_status emr_stream_mode(const void *pack_host, const void *pack_dev, const emr_query *q, const emr_grid *grid,
                           float theta, float band, float w_min, int32_t mode, int32_t types, void *ws,
                           size_t ws_bytes, int64_t chunk_cap, int32_t *h_idx, float *h_w, int64_t cap,
                           int64_t *counts, int64_t *offsets, int64_t timeout_ms, void *stream);

/* ---- fused evaluation without a caller-provided workspace -------------------- */

/* The paper has no counterpart to this call; it exists for callers that cannot
 * allocate device memory themselves (for example a plugin whose host
 * application owns all device memory, or a latency-critical loop that must not
 * incur the implicit device synchronisation of cudaMalloc).
 *
 * Computes exactly what emr_eval_prepare followed by emr_eval_filter computes
 * (same split / band_bits planes, same sparse out entries), but keeps the
 * per-pair records, their scratch and the pair schedule in a static device
 * array owned by libemr: EMR_STATIC_SCRATCH_BYTES (16 MiB) on every GPU that
 * loads the library, held until the process exits. It allocates nothing and
 * calls no allocating routine. The caller still provides the inputs (packed
 * population, query) and the outputs (split, band_bits, out as in
 * emr_eval_filter).
 *
 * Limits and behaviour:
 *  - EMR_ERR_RANGE if the pairs' records do not fit the static array (the size
 *    emr_eval_workspace_size reports must be <= EMR_STATIC_SCRATCH_BYTES);
 *    nothing is launched then.
 *  - The first call on a device looks up the array's device address
 *    (cudaGetSymbolAddress, with that device current) and caches it. With the
 *    CUDA runtime's lazy module loading, that lookup may also be what loads
 *    libemr's device code (and so the array) onto the device; make that first
 *    call before any stream capture.
 *  - All calls on a device share the one array and it keeps the previous
 *    call's contents. The one entry that must start at zero (the pair
 *    schedule's completion counter) is cleared by each call on its stream;
 *    every other entry is written before it is read. Calls whose work overlaps
 *    on the GPU (other streams, other host threads) race on the array:
 *    serialise them.
 * Errors: EMR_ERR_ARG, EMR_ERR_RANGE, EMR_ERR_CUDA. */
#define EMR_STATIC_SCRATCH_BYTES (16u << 20)
emr_status emr_eval_filter_noalloc(const void *pack_host, const void *pack_dev, const emr_query *q,
                                   const emr_grid *grid, float theta, float band, float w_min, uint32_t *split,
                                   uint32_t *band_bits, float *out, void *stream);

/* ---- a6: compaction -------------------------------------------------------- */

/* Bytes of device workspace emr_compact needs for n_pairs pairs. */
emr_status emr_compact_workspace_size(const emr_grid *grid, int32_t n_pairs, size_t *bytes);

/* Per pair, the ascending global indices of the set bits of mask and the CPPN
 * outputs there (the connection list of each (genome, slot)). mask: device
 * uint32 [n_pairs][n_words]; out: device float [n_pairs][n_total] (only the
 * entries at set bits are read). Writes counts (device int64 [n_pairs]),
 * offsets (device int64 [n_pairs + 1], exclusive prefix of counts; offsets[n_pairs]
 * = total), idx (device int32 [cap]) and w (device float [cap], may be NULL):
 * pair r's list is [offsets[r], offsets[r] + counts[r]). Entries at positions
 * >= cap are dropped; compare offsets[n_pairs] with cap after the stream
 * completes. Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY (workspace), EMR_ERR_CUDA. */
emr_status emr_compact(const uint32_t *mask, const float *out, const emr_grid *grid, int32_t n_pairs,
                       int32_t *idx, float *w, int64_t cap, int64_t *counts, int64_t *offsets, void *ws,
                       size_t ws_bytes, void *stream);

/* Same as emr_compact, but the CPPN outputs at the kept positions are
 * recomputed from the per-pair records in eval_ws (prepared by
 * emr_eval_prepare for this pack and query) with the tile kernels' own
 * arithmetic, so the fused path needs no output buffer: the weights equal those
 * emr_eval would have written. mask as from emr_mask_combine; the number of
 * pairs comes from the pack and query. Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY
 * (eval_ws or ws too small), EMR_ERR_CUDA. */
emr_status emr_compact_records(const uint32_t *mask, const void *pack_host, const emr_query *q, const void *eval_ws,
                               size_t eval_ws_bytes, const emr_grid *grid, int32_t *idx, float *w, int64_t cap,
                               int64_t *counts, int64_t *offsets, void *ws, size_t ws_bytes, void *stream);

/* emr_eval_filter (without the output buffer) that also flags, per pair and
 * dense tile, whether any band bit is set: tile_flags is device uint8
 * [n_pairs][n_dense], 1 where the tile holds a band-passing position, else 0.
 * Dense tiles: tile 0 holds depths 0..min(D, 4); tile t >= 1 is the t-th 64 x 64
 * Morton block of depths 5..D in global-index order (n_dense = 1 + the number of
 * such blocks). For emr_select, which reads the planes only in flagged tiles: a
 * pair whose output is constant over the grid (every variance and band value 0)
 * has no flag set, and its rows of split and band_bits are left untouched (use
 * emr_eval_filter where the planes themselves are wanted). Errors as
 * emr_eval_filter. */
emr_status emr_eval_filter_tiles(const void *pack_host, const emr_query *q, const emr_grid *grid, float theta,
                                 float band, float w_min, uint32_t *split, uint32_t *band_bits,
                                 uint8_t *tile_flags, void *ws, size_t ws_bytes, void *stream);

/* Bytes of device workspace emr_select needs for n_pairs pairs (per pair and
 * dense tile: the tile's first list entry and a work item). */
emr_status emr_select_workspace_size(const emr_grid *grid, int32_t n_pairs, size_t *bytes);

/* emr_mask_combine_types followed by emr_compact_records, computed only over the
 * tiles that tile_flags (from emr_eval_filter_tiles) marks: a tile without band
 * bits keeps nothing, whatever its split bits. No mask plane is written. The
 * lists, counts and offsets equal those of the two calls; entries past cap are
 * dropped (compare offsets[n_pairs] with cap). eval_ws: the prepared records;
 * ws: emr_select_workspace_size bytes. Errors: EMR_ERR_ARG, EMR_ERR_CAPACITY
 * (eval_ws or ws), EMR_ERR_RANGE, EMR_ERR_CUDA. */
emr_status emr_select(const uint32_t *split, const uint32_t *band_bits, const uint8_t *tile_flags,
                      const void *pack_host, const emr_query *q, const void *eval_ws, size_t eval_ws_bytes,
                      const emr_grid *grid, int32_t mode, int32_t types, int32_t *idx, float *w, int64_t cap,
                      int64_t *counts, int64_t *offsets, void *ws, size_t ws_bytes, void *stream);

/* Subtree-leaf variance: the split plane under ES-HyperNEAT's reading of a
 * cell's variance (its quadtree measures the spread of the outputs at a
 * region's leaves; the paper's Section 3.2 computes it over a cell's four
 * children, which is the default everywhere else). Cell p of depth d < D
 * splits when the population variance of the outputs at all its depth-D
 * descendants (4^(D - d) positions) exceeds theta. From materialised outputs
 * (out as written by emr_eval); writes the split words of depths 0..D-1 (device
 * uint32 [n_pairs][n_words], position-major), and, when var_out is not NULL,
 * that variance at each position of depths 0..D-1 (device float [n_pairs]
 * [n_total]). Combine with band bits by emr_mask_combine(_types) as usual.
 * ws: emr_subtree_workspace_size bytes (two levels of per-cell aggregates).
 * D at most 11. Errors: EMR_ERR_ARG, EMR_ERR_RANGE, EMR_ERR_CAPACITY,
 * EMR_ERR_CUDA. */
emr_status emr_subtree_workspace_size(const emr_grid *grid, int32_t n_pairs, size_t *bytes);
emr_status emr_subtree_split(const float *out, const emr_grid *grid, int32_t n_pairs, float theta,
                             uint32_t *split, float *var_out, void *ws, size_t ws_bytes, void *stream);

/* HyperNEAT's weight scaling (the indirect encoding of Section 2, where a
 * connection is expressed only when the CPPN output's magnitude exceeds a
 * threshold; the paper's pipeline uses raw outputs, so this is an option) on
 * the weights of lists laid out as emr_compact writes them, in place:
 * w <- sign(w) * w_max * (min(|w|, 1) - w_thr) / (1 - w_thr) when |w| > w_thr,
 * else 0 (combine with w_min = w_thr to drop those entries at discovery).
 * Entries e < min(offsets[n_pairs], cap). Requires 0 <= w_thr < 1, w_max > 0.
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_scale_weights(float *w, const int64_t *offsets, int32_t n_pairs, int64_t cap, float w_thr,
                             float w_max, void *stream);

/* The whole path in one call: emr_eval_prepare, emr_eval_filter_tiles and
 * emr_select on a single workspace that holds the records, the split and band
 * planes, the tile flags and the selection workspace (emr_discover_workspace_
 * size bytes; the planes inside are the library's, not to be read). The pack is
 * planned once. Lists, counts and offsets as emr_select writes them.
 * Errors as the three calls. */
emr_status emr_discover_workspace_size(const void *pack_host, const emr_query *q, const emr_grid *grid,
                                       size_t *bytes);
emr_status emr_discover(const void *pack_host, const void *pack_dev, const emr_query *q, const emr_grid *grid,
                        float theta, float band, float w_min, int32_t mode, int32_t types, void *ws,
                        size_t ws_bytes, int32_t *idx, float *w, int64_t cap, int64_t *counts, int64_t *offsets,
                        void *stream);

/* One asynchronous copy of bytes from src to dst on the stream (host or device
 * memory on either side, told apart by the CUDA runtime's unified addressing):
 * the step's inputs into their device copies and its lists back, without a
 * framework's per-copy overhead. A host buffer must be pinned for the copy to be
 * asynchronous; the caller keeps both buffers alive until the stream has passed
 * the copy. bytes = 0 does nothing. Errors: EMR_ERR_ARG (null pointer with
 * bytes > 0), EMR_ERR_CUDA. */
emr_status emr_copy_async(void *dst, const void *src, size_t bytes, void *stream);

/* Connection type code (0 forward, 1 backward, 2 lateral, 3 self; Section 6
 * taxonomy, see emr_mask_combine_types) of every list entry: type[e] for
 * entries e < min(offsets[n_pairs], cap) of lists laid out as emr_compact
 * writes them (idx: device int32 global indices; offsets: device int64
 * [n_pairs + 1]; type: device uint8 [cap]). n_pairs must be a multiple of q->S.
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_conn_types(const int32_t *idx, const int64_t *offsets, const emr_query *q, const emr_grid *grid,
                          int32_t n_pairs, int64_t cap, uint8_t *type, void *stream);

/* ---- f2: network assembly and the substrate ANN ------------------------------ */

/* Connection cache (Section 7: cached hidden-to-hidden connections make later
 * discovery nearly free). Caller-owned: lists discovered by emr_assemble are
 * kept per (genome content, query slot, query parameters) and reused by later
 * calls for identical genomes (an elite carried to the next generation, or a
 * clone) and slots, up to max_bytes (least recently used entries go first). A
 * genome is identified by its packed records, so any change to it misses.
 * Reuse does not change results: the device path is deterministic. Not
 * thread-safe: one call at a time per cache. Host memory only. create: *cache
 * receives the new cache (NULL on failure); EMR_ERR_ARG (cache NULL),
 * EMR_ERR_ALLOC. destroy: frees the cache and its entries (NULL is a no-op).
 * clear: drops every entry and the counters, keeps max_bytes; EMR_ERR_ARG for
 * NULL. */
typedef struct emr_cache emr_cache;
emr_status emr_cache_create(size_t max_bytes, emr_cache **cache);
emr_status emr_cache_destroy(emr_cache *cache);
emr_status emr_cache_clear(emr_cache *cache);
/* Lookups that hit and missed since creation or the last clear, entries held
 * and their bytes. Any output may be NULL. Errors: EMR_ERR_ARG (cache NULL). */
emr_status emr_cache_stats(const emr_cache *cache, int64_t *hits, int64_t *misses, int64_t *entries,
                           int64_t *bytes);

/* Bytes of device workspace emr_assemble needs (query slots, per-pair records,
 * the three bit planes, compaction workspace and list_cap list entries for
 * max(slots_max, n_in + n_out) slots per genome). */
emr_status emr_assemble_workspace_size(const void *pack_host, int32_t n_in, int32_t n_out, int32_t slots_max,
                                       const emr_grid *grid, int64_t list_cap, size_t *bytes);

/* Build each genome's substrate network (ES-HyperNEAT's construction, which
 * Section 2 summarises and Section 6 configures) with the discovery path of
 * this library for every query:
 *   Phase 1: an outgoing query from each substrate input (in_x, in_y) connects
 *            it to every position it keeps; those positions are hidden nodes.
 *   Phase 2: `rounds` times, an outgoing query from each hidden node found in
 *            the previous round connects it to its kept positions; new
 *            positions join the hidden nodes (0 rounds: feedforward).
 *   Phase 3: an incoming query toward each substrate output (out_x, out_y)
 *            connects the hidden nodes among its kept positions to it.
 *   Pruning: hidden nodes not reachable from an input or not reaching an
 *            output are removed with their connections.
 * Every query uses theta, band, w_min, mode and the connection-type filter
 * types (EMR_CONN_* bits, see emr_substrate_config). Phase 2 queries at most
 * slots_max hidden nodes of a genome at a time (more are taken in further
 * batches); list_cap bounds the entries of one batch.
 * Output (host arrays): genome g has hidden nodes hidden[node_off[g] ..
 * node_off[g+1]) (global grid indices, ascending; emr_index_to_ij gives their
 * coordinates) and connections [conn_off[g], conn_off[g+1]) with source and
 * destination node numbers (inputs 0 .. n_in - 1, outputs n_in .. n_in +
 * n_out - 1, hidden node k at n_in + n_out + k), weight (the CPPN output) and
 * type code (0 forward, 1 backward, 2 lateral, 3 self), sorted by destination
 * then source. cache (optional, NULL for none): query results are looked up
 * there first and added after. Synchronous on `stream`.
 * Errors: EMR_ERR_ARG; EMR_ERR_CAPACITY (workspace too small, a batch's lists
 * exceed list_cap, or hidden_cap / conn_cap too small: node_off and conn_off
 * then hold the true totals); errors of the discovery calls. */
emr_status emr_assemble(const void *pack_host, const void *pack_dev, int32_t n_in, const float *in_x,
                        const float *in_y, int32_t n_out, const float *out_x, const float *out_y,
                        const emr_grid *grid, float theta, float band, float w_min, int32_t mode, int32_t types,
                        int32_t rounds, int32_t slots_max, void *ws, size_t ws_bytes, int64_t list_cap,
                        int64_t *node_off, int32_t *hidden, int64_t hidden_cap, int64_t *conn_off,
                        int32_t *conn_src, int32_t *conn_dst, float *conn_w, uint8_t *conn_type,
                        int64_t conn_cap, emr_cache *cache, void *stream);

/* Forward pass of P assembled networks on K input patterns (device arrays as
 * emr_assemble writes them, copied to the device): input node i holds
 * patterns[k * n_in + i]; every other node starts at 0 and `steps` times all
 * take, at once, the sigmoid 1 / (1 + e^-z) of z = the weighted sum of their
 * sources' previous values (the substrate network of an HyperNEAT-style
 * indirect encoding, Section 2; recurrent connections make the result depend
 * on steps). out[(g * K + k) * n_out + o] receives output o. max_hidden: the
 * largest hidden-node count of a genome (sizes shared memory: the call fails
 * with EMR_ERR_RANGE when 8 (n_in + n_out + max_hidden) K bytes do not fit).
 * Errors: EMR_ERR_ARG, EMR_ERR_RANGE, EMR_ERR_CUDA. */
emr_status emr_ann_forward(int32_t P, int32_t n_in, int32_t n_out, int32_t max_hidden, const int64_t *node_off,
                           const int64_t *conn_off, const int32_t *conn_src, const int32_t *conn_dst,
                           const float *conn_w, int32_t K, const float *patterns, int32_t steps, float *out,
                           void *stream);

/* ---- misc -------------------------------------------------------------------- */

/* Static description of a status code. */
const char *emr_strerror(emr_status status);

/* Library version: major * 10000 + minor * 100 + patch. */
int32_t emr_version(void);

#ifdef __cplusplus
}
#endif

#endif /* EMR_H */
