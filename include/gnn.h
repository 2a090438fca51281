/*
 * gnn.h -- C ABI of the GB300 interaction-network edge classifier.
 *
 * The library scores candidate edges of a particle-detector hit graph with an
 * interaction network, the edge-classification stage of the GNN tracking
 * pipeline (paper Section 2.1: space points and the candidate edges built
 * between them go in; the interaction network gives every edge a score that
 * the connected-components step thresholds into track candidates).  The
 * paper's service boundary takes a 2-D array of space points (rows) by raw
 * features (columns) (Section 2.3); this ABI keeps that layout and adds the
 * candidate edges, and returns one score per edge.
 *
 * Network (fp32 model; every MLP is L x [Linear -> LayerNorm -> ReLU]):
 *   h_j  = MLP_node_encoder(x_j)            e_ij = MLP_edge_encoder(dr, dphi)
 *   T times: m_ij = MLP_edge([h_i, h_j, e_ij]);  e_ij = m_ij
 *            a_j  = sum over edges (i -> j) of m_ij
 *            h_j  = MLP_node([h_j, a_j])
 *   score_ij = sigmoid(w_o . MLP_classifier([h_i, h_j, e_ij]) + b_o)
 * with dr = x_j[0] - x_i[0] and dphi = x_j[1] - x_i[1] wrapped into (-1, 1]
 * (columns 0 and 1 hold r/1000 and phi/pi).
 *
 * Threading and streams: every call that takes a stream only enqueues work on
 * it (no host synchronisation) unless stated otherwise.  A context is not
 * safe for concurrent use from several streams or threads (it owns one
 * workspace); use one context per stream.
 *
 * Return codes: GNN_OK (0) or a negative gnn_status_code.  Errors found on
 * the host are returned at once; errors found by the kernels are recorded in
 * the context's device error word and returned by gnn_status().
 */
#ifndef GNN_GB300_H
#define GNN_GB300_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* gnn_stream_t; /* a cudaStream_t; NULL = legacy default stream */

/* The largest count any call accepts (nodes, edges, an output capacity): 2^31 - 1 - 8192, so that
 * the kernels' 32-bit row indices stay in range after rounding up to whole blocks and tiles.  A
 * larger count (or a negative one) is INVALID_ARG, returned before any device work. */
#define GNN_MAX_COUNT 2147475455

enum gnn_status_code {
  GNN_OK = 0,
  GNN_ERR_INVALID_ARG = -1,    /* null pointer, bad size or unsupported configuration */
  GNN_ERR_BAD_WEIGHTS = -2,    /* weight blob: wrong magic/version/size or config mismatch */
  GNN_ERR_OOM = -3,            /* device allocation failed */
  GNN_ERR_CUDA = -4,           /* a CUDA runtime call or kernel launch failed */
  GNN_ERR_INDEX_RANGE = -5,    /* device: an edge endpoint was outside [0, n_nodes) */
  GNN_ERR_DEVICE_TIMEOUT = -6, /* device: a pipeline wait expired; results are invalid */
  GNN_ERR_CAPACITY = -7,       /* device: an output buffer was too small (gnn_build_graph) */
};

enum gnn_precision {
  GNN_PRECISION_FP32 = 0,      /* fp32 weights and state; products as three bf16 pieces */
  GNN_PRECISION_BF16 = 1,      /* bf16 weights, activations and stored states (h, e, a); fp32
                                  accumulation and LayerNorm; the blob's values must be bf16 */
};

/* Model configuration (must equal the blob header). */
typedef struct gnn_config {
  int32_t version;             /* must be 1 */
  int32_t n_node_feat;         /* F_n: node feature columns, 2..16 (cols 0, 1 = r/1000, phi/pi) */
  int32_t n_edge_feat;         /* must be 2: (dr, dphi) */
  int32_t hidden;              /* H: 64 or 128 */
  int32_t n_iters;             /* T: message-passing iterations, 0..64 */
  int32_t mlp_layers;          /* L: Linear layers per MLP, 2..4 */
  int32_t precision;           /* enum gnn_precision */
  float ln_eps;                /* LayerNorm epsilon (1e-5) */
} gnn_config;

typedef struct gnn_ctx gnn_ctx;

/*
 * gnn_create -- build a context on the current CUDA device.
 *
 * weights_host: host pointer to a little-endian weight blob of weights_bytes
 * bytes: a header of eight int32 (magic 0x57474E47, version 1, n_node_feat,
 * n_edge_feat, hidden, n_iters, mlp_layers, precision), float32 ln_eps, int32
 * reserved, int64 float count; then float32 arrays.  For each MLP in the order
 * node_encoder, edge_encoder, edge_network, node_network, edge_classifier and
 * each of its L layers: W [H, in] row-major, b [H], gamma [H], beta [H]
 * (in = F_n, 2, 3H, 2H, 3H for layer 1, H afterwards; the 3H inputs are
 * ordered [h_src, h_dst, e] and the 2H input [h, a]); then w_o [H] and b_o [1].
 * The blob is copied and repacked; the caller may free it on return.
 * On success *out receives the context (free with gnn_destroy).
 * Errors: INVALID_ARG (null pointer, unsupported config), BAD_WEIGHTS, OOM,
 * CUDA.  Synchronous.
 */
int gnn_create(const gnn_config* cfg, const void* weights_host, size_t weights_bytes, gnn_ctx** out);

/*
 * gnn_reserve -- size the context's workspace for graphs up to max_nodes
 * nodes and max_edges edges, so that later gnn_infer calls of that size
 * allocate nothing.  Synchronous (device allocation).  Errors: INVALID_ARG,
 * OOM.
 */
int gnn_reserve(gnn_ctx* ctx, int64_t max_nodes, int64_t max_edges);

/*
 * gnn_infer -- score every edge of one graph (a single event, or several
 * events concatenated block-diagonally).
 *
 *   node_feats  device, float32 [n_nodes, n_node_feat] row-major, 16-byte aligned
 *   edge_index  device, int32 [2, n_edges] row-major: row 0 = source ids,
 *               row 1 = destination ids, any order; duplicates and
 *               self-loops are legal
 *   edge_scores device, float32 [n_edges]: score of edge k of the input order
 *
 * All three buffers are caller-owned and must stay valid until the stream
 * reaches this work; the library never frees them.  n_edges == 0 is a no-op;
 * n_nodes == 0 with n_edges > 0 and sizes above GNN_MAX_COUNT are
 * INVALID_ARG.  The workspace grows here (synchronous allocation) when the
 * graph is larger than any earlier one; call gnn_reserve first to avoid it.
 * An edge with an endpoint outside [0, n_nodes) gets a NaN score, takes no
 * part in any aggregation, and makes gnn_status report INDEX_RANGE.
 * Scores are deterministic: the same inputs give bitwise-identical outputs.
 */
int gnn_infer(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
              int64_t n_edges, float* edge_scores, gnn_stream_t stream);

/*
 * gnn_infer_host -- gnn_infer on HOST buffers (the form a serving backend
 * receives requests in): copies node_feats [n_nodes, n_node_feat] float32 and
 * edge_index [2, n_edges] int32 from host memory into the context's staging
 * buffers, scores on the device, copies the scores back into edge_scores
 * [n_edges] float32 (host), and synchronises `stream` before returning.
 * Pinned (page-locked) host memory makes the copies asynchronous DMA;
 * pageable memory also works.  Same argument rules and errors as gnn_infer,
 * plus the device status of this call (as gnn_status would return it).
 */
int gnn_infer_host(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
                   int64_t n_edges, float* edge_scores, gnn_stream_t stream);

/*
 * gnn_embed_load -- load the embedding MLP (paper Section 2.1: the first step maps every space
 * point's raw features into a latent space where hits of one track lie close together).  Network:
 * y = normalize(W_out . MLP_L(x) + b_out), L hidden layers Linear -> LayerNorm -> ReLU of the
 * context's hidden width, then a Linear to D outputs, scaled to unit length (a zero vector stays
 * zero).  Blob (little-endian, copied): eight int32 (magic 0x4D454E47 "GNEM", version 1,
 * n_node_feat, hidden, L (2..4), precision, D (1..16), reserved), float32 ln_eps, int32 reserved,
 * int64 float count, then per hidden layer W [H, in] row-major, b, gamma, beta (in = n_node_feat
 * for layer 1, H afterwards), then W_out [D, H], b_out [D].  n_node_feat, hidden and precision
 * must equal the context's.  A later call replaces it.  Errors: INVALID_ARG, BAD_WEIGHTS, OOM, CUDA.
 *
 * gnn_embed -- embedding of every hit: node_feats device float32 [n_nodes, n_node_feat] in,
 * embedding device float32 [n_nodes, D] out (caller-owned).  Enqueued on `stream`.  Errors:
 * INVALID_ARG (no embedding loaded, null pointer, bad size), CUDA.
 *
 * gnn_build_graph -- candidate edges by fixed-radius neighbours in the embedding space (Section
 * 2.1: the graph is built between hits closer than a radius in the latent space).  Every pair of
 * hits whose squared distance, summed over the emb_dim coordinates in order in fp32 with one
 * rounding per product and per sum, is below radius * radius (rounded to fp32) becomes one edge,
 * oriented from the hit with the smaller r (node_feats column 0; the smaller id on a tie).
 *   embedding  device float32 [n_nodes, emb_dim], emb_dim 1..16; unit vectors (as gnn_embed
 *              writes them) are searched on a grid over [-1, 1]^K (K = 4 for emb_dim >= 4,
 *              else 3), other values stay exact but
 *              crowd into the grid's edge cells
 *   node_feats device float32 [n_nodes, n_node_feat] (column 0 orients the edges)
 *   edge_index device int32 with room for [2, max_edges], output: contiguous [2, n_edges]
 *   n_edges    device int32 [1], output: the number of edges found
 * When n_edges exceeds max_edges nothing is written to edge_index, *n_edges still holds the
 * count (saturated at INT32_MAX), and gnn_status reports GNN_ERR_CAPACITY: call again with room
 * for that many.  The order
 * of the edges is deterministic.  Uses a scratch buffer of the context (grown on demand,
 * synchronous then): besides the sorted copies, 128 bytes per hit for the partner chains the
 * counting pass keeps (see gnn_debug_graph_pool).  Errors: INVALID_ARG (radius <= 0, emb_dim out
 * of range, null pointer, bad sizes), OOM, CUDA.
 */
int gnn_embed_load(gnn_ctx* ctx, const void* weights_host, size_t weights_bytes);
int gnn_embed(gnn_ctx* ctx, const float* node_feats, int64_t n_nodes, float* embedding, gnn_stream_t stream);
int gnn_build_graph(gnn_ctx* ctx, const float* embedding, int emb_dim, const float* node_feats, int64_t n_nodes,
                    float radius, int64_t max_edges, int32_t* edge_index, int32_t* n_edges, gnn_stream_t stream);

/*
 * gnn_filter_load -- load the filtering MLP (paper Section 2.1: the step before the GNN scores every
 * candidate edge from the raw features of its two hits; applyFiltering then drops the edges below
 * a fixed threshold).  Network: s = sigmoid(w_o . MLP_L([x_src, x_dst]) + b_o), each of its L
 * layers Linear -> LayerNorm -> ReLU, in the context's precision and hidden width.
 * Blob (little-endian, copied; the caller may free it): eight int32 (magic 0x4C464E47 "GNFL",
 * version 1, n_node_feat, hidden, mlp_layers (2..4), precision, two reserved), float32 ln_eps,
 * int32 reserved, int64 float count, then float32 arrays: per layer W [H, in] row-major, b, gamma,
 * beta (in = 2 * n_node_feat for layer 1, H afterwards), then w_o [H], b_o [1].  n_node_feat,
 * hidden and precision must equal the context's.  A later call replaces the filter.
 * Errors: INVALID_ARG, BAD_WEIGHTS, OOM, CUDA.  Synchronous.
 *
 * gnn_filter_edges -- score every candidate edge with the filtering MLP and keep those with
 * score > threshold, in input order.
 *   node_feats  device float32 [n_nodes, n_node_feat]
 *   edge_index  device int32 [2, n_edges] (row 0 sources, row 1 destinations)
 *   edge_scores device float32 [n_edges], output: filter score of every input edge (NaN for an edge
 *               with an endpoint out of range, which is never kept; gnn_status then reports
 *               INDEX_RANGE)
 *   kept_index  device int32 with room for [2, n_edges], output: the kept edges as a contiguous
 *               [2, n_kept] edge index (row 1 starts at n_kept), ready for gnn_infer
 *   kept_id     device int32 [n_edges] or NULL, output: input id of every kept edge
 *   n_kept      device int32 [1], output
 * All buffers are caller-owned.  Enqueued on `stream`; uses the context's workspace (it may grow,
 * as in gnn_infer).  Errors: INVALID_ARG (no filter loaded, null pointer, bad sizes), OOM, CUDA.
 */
int gnn_filter_load(gnn_ctx* ctx, const void* weights_host, size_t weights_bytes);
int gnn_filter_edges(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
                     int64_t n_edges, float threshold, float* edge_scores, int32_t* kept_index, int32_t* kept_id,
                     int32_t* n_kept, gnn_stream_t stream);

/*
 * gnn_track_labels -- track candidates from scored edges: one integer label per hit.  The
 * edge-classification scores are thresholded and the weakly connected components of the kept
 * edges are the track candidates (paper Section 2.1, the step after the interaction network);
 * the service returns an integer label per space point (Section 2.3).
 *
 *   edge_scores device float32 [n_edges], input edge order (as gnn_infer writes them)
 *   edge_index  device int32 [2, n_edges]: row 0 sources, row 1 destinations
 *   threshold   an edge is kept when its score is > threshold (NaN scores are never kept)
 *   labels      device int32 [n_nodes], output: the smallest node id of the hit's component
 *               (a hit without kept edges is its own component); caller-owned
 *
 * Edges with an endpoint outside [0, n_nodes) are skipped.  The labels do not depend on thread
 * or edge order.  Enqueued on `stream`; uses no workspace (the labels array is the union-find
 * forest).  Every union and find loop gives up after 1 s of wall-clock time (%globaltimer) and
 * then records GNN_ERR_DEVICE_TIMEOUT in the context's device error word (see gnn_status); the
 * labels are then invalid.  Errors: INVALID_ARG (null pointer, negative sizes or sizes above
 * GNN_MAX_COUNT, n_nodes == 0 with edges), CUDA.
 */
int gnn_track_labels(gnn_ctx* ctx, const float* edge_scores, const int32_t* edge_index, int64_t n_nodes,
                     int64_t n_edges, float threshold, int32_t* labels, gnn_stream_t stream);

/*
 * gnn_profile_enable -- when on != 0, later gnn_infer / gnn_infer_host calls
 * record a CUDA event pair on their stream around every kernel group, so
 * gnn_profile_read can report device time per group.  Off by default.
 *
 * gnn_profile_read -- synchronise the recorded events and write, for each
 * group g < n_groups, the summed device milliseconds ms[g] and the number of
 * kernel launches launches[g]; then clear the records.  Groups: 0 CSR build
 * (all its kernels), 1 node encoder, 2 edge encoder, 3 edge update, 4 node
 * update, 5 classifier, 6 host<->device copies of gnn_infer_host, 7 message
 * aggregation, 8 filtering MLP, 9 embedding MLP.  Either output pointer may
 * be NULL.  Returns the number of groups (10) or an error.
 */
int gnn_profile_enable(gnn_ctx* ctx, int on);
int gnn_profile_read(gnn_ctx* ctx, double* ms, int64_t* launches, int n_groups);

/*
 * gnn_status -- synchronise `stream`, then return and clear the device error
 * word of the context: GNN_OK, GNN_ERR_INDEX_RANGE, GNN_ERR_DEVICE_TIMEOUT,
 * GNN_ERR_CAPACITY (gnn_build_graph) or GNN_ERR_CUDA (a failed synchronisation).
 */
int gnn_status(gnn_ctx* ctx, gnn_stream_t stream);

/* gnn_destroy -- wait for the device (cudaDeviceSynchronize: the context does not know which
 * streams used it, so other work on the device is waited for too) and free ctx and all its
 * device memory. NULL is a no-op. */
void gnn_destroy(gnn_ctx* ctx);

/* gnn_error_string -- static text for a status code. */
const char* gnn_error_string(int code);

/*
 * gnn_debug_copy -- test hook: copy an internal buffer of the last gnn_infer
 * into caller device memory `dst` of at least `bytes` bytes (enqueued on
 * `stream`).  which: 0 rowptr int32 [N+1], 1 perm int32 [E] (CSR slot ->
 * input edge id), 2 src_sorted int32 [E], 3 node state h, 4 edge state e (CSR
 * order).  The states are float32 (bfloat16 for GNN_PRECISION_BF16) in the row-tiled layout of the kernels:
 * R = rows rounded up to a multiple of 128, element (r, c) at index
 * ((r / 128) * (H / 16) + bp) * 2048 + (r % 128) * 16 + x, R * H floats, where
 * b = c / 8, bp = b / 2 and x = 4 * ((c % 8) / 2) + 2 * (b % 2) + c % 2.
 * Errors: INVALID_ARG when the buffer is unknown or `bytes` is too small.
 */
int gnn_debug_copy(gnn_ctx* ctx, int which, void* dst, size_t bytes, gnn_stream_t stream);

/*
 * Failure-injection hooks for tests (no paper counterpart).  Neither faults nor hangs a GPU.
 *
 * gnn_debug_fail_allocs -- the next n device allocations made by the library (context creation,
 * workspace growth, gnn_infer_host staging) fail as if the device were out of memory, so the
 * GNN_ERR_OOM paths can be exercised; n = 0 cancels.  Process-wide.  Errors: INVALID_ARG (n < 0).
 *
 * gnn_debug_wait_timeout -- enqueue on `stream` one kernel that waits, through the same bounded
 * wait every pipeline wait in the library uses, on an mbarrier that nothing completes; after
 * limit_ns nanoseconds (0 < limit_ns <= 2e9) the wait gives up and records GNN_ERR_DEVICE_TIMEOUT
 * in the context's device error word, which gnn_status then returns (and clears).  The context
 * stays usable.  Errors: INVALID_ARG, CUDA.
 */
int gnn_debug_fail_allocs(int n);
int gnn_debug_wait_timeout(gnn_ctx* ctx, int64_t limit_ns, gnn_stream_t stream);

/*
 * gnn_debug_graph_pool -- test hook for gnn_build_graph (no paper counterpart).  The counting pass
 * keeps every hit's partners in a chain of 15-entry chunks, the hit's own first chunk plus chunks
 * from a pool, and the writing pass copies them; a hit whose chain could not grow because the pool
 * was used up is searched again instead, with the same result.  This sets the pool size in chunks
 * for later calls on this context (0: every hit with more than 15 partners takes the search-again
 * path); a negative value restores the default of one pool chunk per hit.  Errors: INVALID_ARG
 * (null context).
 */
int gnn_debug_graph_pool(gnn_ctx* ctx, int64_t chunks);

/*
 * gnn_csr_build_noalloc -- the destination-keyed CSR of an edge list, built
 * without allocating any device memory.  (Library plumbing: the paper has no
 * counterpart.)  It is for callers that must not allocate: a serving backend
 * or host framework whose memory planner owns every device allocation and
 * forbids new ones after start-up, or code that must keep cudaMalloc and
 * cudaFree (and their implicit device synchronisation) off its request path.
 *
 * Scratch is one fixed, library-owned device array of
 * GNN_CSR_NOALLOC_SCRATCH_BYTES bytes, allocated when the library is loaded
 * on a device and held by every device that loads the library until the
 * process exits.  The caller provides only inputs and outputs:
 *   edge_index device int32 [2, n_edges] (row 0 sources, row 1 destinations)
 *   rowptr     device int32 [n_nodes + 1]: first sorted slot of each node
 *   perm       device int32 [n_edges]: input edge id of each sorted slot
 *   src_sorted device int32 [n_edges]: source of each sorted slot
 * The result is bit-identical to the CSR gnn_infer builds: edges stably
 * sorted by destination (ties keep input order).  Edges with an endpoint
 * outside [0, n_nodes) are placed after rowptr[n_nodes], in input order,
 * with source 0: rowptr[n_nodes] < n_edges is the only signal of them (this
 * call has no context, so no error word records them).
 * Limits: n_edges <= GNN_CSR_NOALLOC_MAX_EDGES and 0 <= n_nodes <= GNN_MAX_COUNT;
 * larger sizes, negative sizes or null pointers return GNN_ERR_INVALID_ARG
 * before any device work.  Every call looks up the scratch array's device
 * address in the current context (cudaGetSymbolAddress: it allocates and
 * enqueues nothing, and follows the array when a device reset or another
 * context gives it a new address); the first call in a context may load the
 * library's device code, so make that first call outside any stream capture.
 * All calls share the one array and it keeps the last
 * call's contents (nothing in it needs to start at zero); calls that overlap
 * on the GPU (several streams, or several host threads) race on it and must
 * be serialised by the caller.  Enqueued on `stream`; no host synchronisation.
 * Errors: INVALID_ARG, CUDA.
 */
#define GNN_CSR_NOALLOC_MAX_EDGES (1 << 20)
#define GNN_CSR_NOALLOC_SCRATCH_BYTES (5u * 4u * GNN_CSR_NOALLOC_MAX_EDGES + 4u * 256u * 256u)
int gnn_csr_build_noalloc(const int32_t* edge_index, int64_t n_nodes, int64_t n_edges, int32_t* rowptr,
                          int32_t* perm, int32_t* src_sorted, gnn_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* GNN_GB300_H */
