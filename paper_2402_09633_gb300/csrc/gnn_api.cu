// C ABI and host orchestration of the interaction-network edge classifier.
//
// gnn_create parses the weight blob and repacks every H x H weight block into
// the layout the tensor-core kernels read straight into shared memory
// (bf16 hi and lo parts, K-major rows of 128 bytes, 128-byte swizzle).  The
// first Linear layer of the edge network and of the classifier acts on
// [h_src, h_dst, e]; it is split into three H x H blocks W_s, W_d, W_e so that
//   W1 [h_src; h_dst; e] + b1 = (W_s h_src) + (W_d h_dst + b1) + W_e e,
// where the two node terms are computed once per node (projections P_s, P_d)
// instead of once per edge.  The node network's first layer on [h, a] is
// split the same way into W_h and W_a.
//
// gnn_infer enqueues: CSR build (validate, radix sort by destination, gather,
// row pointers) -> node encoder (+ projections) -> edge encoder -> T x (edge
// update, node update with aggregation + projections) -> classifier.
#include <cuda_runtime.h>
#include <algorithm>
#include <atomic>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <utility>
#include <vector>

#include "../../include/gnn.h"
#include "compact.cuh"
#include "components.cuh"
#include "csr.cuh"
#include "frnn.cuh"
#include "mlp_tiles.cuh"

using namespace gnn;

namespace {

constexpr uint32_t kBlobMagic = 0x57474E47u;
constexpr uint32_t kFilterMagic = 0x4C464E47u;   // "GNFL": the filtering MLP's weight blob
constexpr uint32_t kEmbedMagic = 0x4D454E47u;    // "GNEM": the embedding MLP's weight blob
constexpr int kHeaderBytes = 8 * 4 + 4 + 4 + 8;

struct Layer { const float* W; const float* b; const float* g; const float* be; int in; };

enum Mlp { NODE_ENC = 0, EDGE_ENC = 1, EDGE_NET = 2, NODE_NET = 3, CLASSIFIER = 4, N_MLP = 5 };

struct KernelPlan {          // job list and parameter vectors of one tile-kernel launch
  int n_jobs = 0;
  int job_mat[kMaxJobs] = {0};
  int job_acc[kMaxJobs] = {0};
  std::vector<float> vecs;
  float* d_vecs = nullptr;
  const uint8_t* wmats = nullptr;   // its weight matrices (null: the context's)
};

}  // namespace

struct gnn_ctx {
  gnn_config cfg;
  int device = 0;
  int n_sm = 0;
  uint8_t* d_mats = nullptr;       // packed weight matrices
  uint32_t mat_bytes = 0;
  // plans: 0 node enc -> edge net, 1 node enc -> classifier, 2 edge enc,
  //        3 edge update, 4 node update -> edge net, 5 node update -> classifier, 6 classifier
  KernelPlan plan[7];
  // filtering step (gnn_filter_load): plan, packed deep-layer matrices, layers, LayerNorm eps
  KernelPlan filter_plan;
  uint8_t* d_filter_mats = nullptr;
  int filter_layers = 0;
  float filter_eps = 0.f;
  // embedding step (gnn_embed_load) and graph building scratch
  KernelPlan embed_plan;
  uint8_t* d_embed_mats = nullptr;
  int embed_layers = 0, embed_dim = 0;
  float embed_eps = 0.f;
  int* aux = nullptr;
  size_t aux_ints = 0;
  int64_t graph_pool = -1;             // graph building: pool chunks for partner chains (-1: one per hit)
  uint32_t* d_err = nullptr;
  // workspace
  void* ws = nullptr;
  int64_t cap_nodes = -1, cap_edges = -1;
  int *keys_a = nullptr, *keys_b = nullptr, *vals_a = nullptr, *vals_b = nullptr, *src_c = nullptr;
  int *hist = nullptr, *perm = nullptr, *src_sorted = nullptr, *dst_sorted = nullptr, *rowptr = nullptr;
  int* key_sorted = nullptr;
  void *e = nullptr, *h = nullptr, *agg = nullptr;  // stored states (fp32 or bf16 per precision)
  float *ps = nullptr, *pd = nullptr;
  int64_t last_nodes = 0, last_edges = 0;
  // staging for gnn_infer_host
  void* stage = nullptr;
  size_t stage_bytes = 0;
  // profiling: event pairs around kernel groups
  struct ProfRec { int group; int launches; cudaEvent_t a, b; };
  bool prof_on = false;
  std::vector<ProfRec> prof;
  size_t prof_used = 0;
#ifdef GNN_TRACE
  unsigned long long* trace = nullptr;   // stamps of CTA 0 of the traced kernel kind
  int trace_kind = -1;
#endif
};

namespace {

inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}
inline float bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

// Byte offset of element (n, k) of an H x H block in the K-major, 128-byte
// swizzled layout: 64-column chunks, 8-row atoms of 1024 bytes, 16-byte units
// of a row permuted by XOR with the row index inside the atom.
inline size_t swizzled_offset(int H, int n, int k) {
  const int kc = k / 64, kk = k % 64;
  return (size_t)kc * (H * 128) + (size_t)(n / 8) * 1024 + (n % 8) * 128 +
         (((kk / 8) ^ (n % 8)) * 16) + (kk % 8) * 2;
}

// Pack columns [col0, col0+H) of W [H, ld] into hi/lo bf16 parts (fp32 model), or
// into the single bf16 part (bf16 model: W holds bf16 values, hi == W exactly).
void pack_block(const float* W, int ld, int col0, int H, bool with_lo, uint8_t* out) {
  const size_t part = (size_t)H * H * 2;
  for (int n = 0; n < H; ++n)
    for (int k = 0; k < H; ++k) {
      const float v = W[(size_t)n * ld + col0 + k];
      const uint16_t hi = f32_to_bf16_rne(v);
      const size_t off = swizzled_offset(H, n, k);
      std::memcpy(out + off, &hi, 2);
      if (with_lo) {
        const uint16_t lo = f32_to_bf16_rne(v - bf16_to_f32(hi));
        std::memcpy(out + part + off, &lo, 2);
      }
    }
}

void push(std::vector<float>& v, const float* p, size_t n) { v.insert(v.end(), p, p + n); }

// W' = (I - 11^T/H) W and b' = b - mean(b): the LayerNorm after the layer then sees a
// zero-mean pre-activation (the fp32 model's kernels compute only the variance).
void centre_layer(const float* W, const float* b, int H, int in, std::vector<float>& Wc, std::vector<float>& bc) {
  Wc.resize((size_t)H * in);
  bc.resize(H);
  for (int k = 0; k < in; ++k) {
    double mu = 0.0;
    for (int n = 0; n < H; ++n) mu += W[(size_t)n * in + k];
    mu /= H;
    for (int n = 0; n < H; ++n) Wc[(size_t)n * in + k] = (float)(W[(size_t)n * in + k] - mu);
  }
  double mb = 0.0;
  for (int n = 0; n < H; ++n) mb += b[n];
  mb /= H;
  for (int n = 0; n < H; ++n) bc[n] = (float)(b[n] - mb);
}

// Every whole H-float segment of a plan's vector block is one per-column vector (bias, gamma,
// beta, head weights, a first-layer weight row); the kernels read them in block-pair order:
// column 8b + 2q + e at 16*(b/2) + 4q + 2*(b%2) + e.  A trailing partial segment (the head
// bias) stays as is.  Then padded to 16 bytes.
void finish_vecs(std::vector<float>& v, int H) {
  std::vector<float> seg(H);
  for (size_t base = 0; base + H <= v.size(); base += H) {
    for (int q = 0; q < 4; ++q)
      for (int b = 0; b < H / 8; ++b)
        for (int e = 0; e < 2; ++e) seg[16 * (b / 2) + 4 * q + 2 * (b % 2) + e] = v[base + 8 * b + 2 * q + e];
    std::copy(seg.begin(), seg.end(), v.begin() + base);
  }
  v.resize(padded_vec_floats((int)v.size()), 0.f);
}

// Test hook: the next g_fail_allocs device allocations made by the library fail (host-side fault
// injection for the allocation-failure paths; see gnn_debug_fail_allocs).
std::atomic<int> g_fail_allocs{0};

cudaError_t dev_alloc(void** p, size_t bytes) {
  int n = g_fail_allocs.load();
  while (n > 0 && !g_fail_allocs.compare_exchange_weak(n, n - 1)) {
  }
  if (n > 0) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(p, bytes);
}

// A kernel that waits, through the library's bounded wait, on an mbarrier nothing arrives on.
__global__ void wait_timeout_kernel(uint64_t limit_ns, uint32_t* err) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  abort_flag = 0;
  fence_mbar_init();
  bounded_wait(&bar, 0, &abort_flag, err, limit_ns);
}

int cuda_fail(cudaError_t e) {
  (void)cudaGetLastError();
  return e == cudaErrorMemoryAllocation ? GNN_ERR_OOM : GNN_ERR_CUDA;
}

// Every count a call accepts (nodes, edges, output capacity) lies in [0, GNN_MAX_COUNT], so that
// the kernels' 32-bit row indices stay in range after rounding up to a whole block or radix tile
// (at most 8192 rows).
inline bool count_ok(int64_t n) { return n >= 0 && n <= (int64_t)GNN_MAX_COUNT; }

// Blocks of `per_block` threads (or rows) covering n, computed in 64 bits.
inline unsigned blocks_for(int64_t n, int64_t per_block) { return (unsigned)((n + per_block - 1) / per_block); }

// Launch as a programmatic dependent of the previous kernel in the stream: the kernel may start
// while that one finishes its last CTAs, and waits for it (pdl_wait) before touching its data.
// Every kernel launched this way calls pdl_wait before its first access to data an earlier
// kernel writes.  Returns the launch status.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), unsigned grid, unsigned block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

constexpr int kProfGroups = 10;

// Returns the record index, or -1 when profiling is off.
int prof_begin(gnn_ctx* c, int group, int launches, cudaStream_t st) {
  if (!c->prof_on) return -1;
  if (c->prof_used == c->prof.size()) {
    gnn_ctx::ProfRec r{};
    if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return -1;
    c->prof.push_back(r);
  }
  gnn_ctx::ProfRec& r = c->prof[c->prof_used];
  r.group = group;
  r.launches = launches;
  cudaEventRecord(r.a, st);
  return (int)c->prof_used++;
}
void prof_end(gnn_ctx* c, int idx, cudaStream_t st) {
  if (idx >= 0) cudaEventRecord(c->prof[idx].b, st);
}

template <TileKind K, int H, bool BF>
cudaError_t set_smem_attr() {
  return cudaFuncSetAttribute(mlp_tile_kernel<K, H, BF>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              227 * 1024);
}

template <int H, bool BF>
cudaError_t set_all_attrs() {
  cudaError_t e;
  if ((e = set_smem_attr<TileKind::NodeEncoder, H, BF>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<TileKind::EdgeEncoder, H, BF>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<TileKind::EdgeUpdate, H, BF>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<TileKind::NodeUpdate, H, BF>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<TileKind::Filter, H, BF>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<TileKind::Embed, H, BF>()) != cudaSuccess) return e;
  return set_smem_attr<TileKind::Classifier, H, BF>();
}

template <TileKind K, int H, bool BF>
cudaError_t launch_tile(gnn_ctx* c, const KernelPlan& pl, TileParams p, cudaStream_t st) {
  p.n_jobs = pl.n_jobs;
  for (int j = 0; j < kMaxJobs; ++j) { p.job_mat[j] = pl.job_mat[j]; p.job_acc[j] = pl.job_acc[j]; }
  p.vecs = pl.d_vecs;
  p.n_vec_floats = (int)pl.vecs.size();
  p.wmats = pl.wmats ? pl.wmats : c->d_mats;
  p.mat_bytes = c->mat_bytes;
  p.n_tiles = (p.n_rows + kTileRows - 1) / kTileRows;
  if (p.n_tiles == 0) return cudaSuccess;
  const uint32_t smem = tile_launch_smem<H, BF>(p.n_vec_floats);
  const int grid = tile_grid(p.n_tiles, c->n_sm);
#ifdef GNN_TRACE
  p.trace = ((int)K == c->trace_kind) ? c->trace : nullptr;
#endif
  static const int group[7] = {1, 2, 3, 4, 5, 8, 9};   // NodeEncoder, EdgeEncoder, EdgeUpdate, NodeUpdate, Classifier, Filter, Embed
  const int pr = prof_begin(c, group[(int)K], 1, st);
  const cudaError_t err = launch_pdl(mlp_tile_kernel<K, H, BF>, grid, kThreads, smem, st, p);
  prof_end(c, pr, st);
  return err;
}

template <int H, bool BF>
int run_network(gnn_ctx* c, const float* x, int N, int E, float* scores, cudaStream_t st) {
  TileParams p{};
  p.n_nodes = N;
  p.n_layers = c->cfg.mlp_layers;
  p.eps = c->cfg.ln_eps;
  p.x = x;
  p.x_stride = c->cfg.n_node_feat;
  p.src_sorted = c->src_sorted;
  p.dst_sorted = c->dst_sorted;
  p.key_sorted = c->key_sorted;
  p.perm = c->perm;
  p.rowptr = c->rowptr;
  p.e = c->e; p.h = c->h; p.ps = c->ps; p.pd = c->pd; p.agg = c->agg;
  p.scores = scores;
  p.err = c->d_err;
  const int T = c->cfg.n_iters;

  cudaError_t le = cudaSuccess;                        // first launch error
  auto chk = [&](cudaError_t e) { if (le == cudaSuccess) le = e; };
  TileParams pn = p; pn.n_rows = N; pn.n_feat = c->cfg.n_node_feat;
  chk(launch_tile<TileKind::NodeEncoder, H, BF>(c, c->plan[T > 0 ? 0 : 1], pn, st));
  TileParams pe = p; pe.n_rows = E; pe.n_feat = 2;
  chk(launch_tile<TileKind::EdgeEncoder, H, BF>(c, c->plan[2], pe, st));
  for (int t = 1; t <= T; ++t) {
    chk(launch_tile<TileKind::EdgeUpdate, H, BF>(c, c->plan[3], pe, st));
    {
      const int pr = prof_begin(c, 7, 1, st);
      chk(launch_pdl(aggregate_kernel<H, BF>, blocks_for(N, agg_nodes_per_block<H>()), 256, 0, st, (const void*)c->e,
                     (const int*)c->rowptr, N, c->agg));
      prof_end(c, pr, st);
    }
    chk(launch_tile<TileKind::NodeUpdate, H, BF>(c, c->plan[t < T ? 4 : 5], pn, st));
  }
  chk(launch_tile<TileKind::Classifier, H, BF>(c, c->plan[6], pe, st));
  const cudaError_t err = le != cudaSuccess ? le : cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

int64_t state_bytes(const gnn_ctx* c) { return c->cfg.precision == GNN_PRECISION_BF16 ? 2 : 4; }

void free_workspace(gnn_ctx* c) {
  if (c->ws) cudaFree(c->ws);
  c->ws = nullptr;
  c->cap_nodes = c->cap_edges = -1;
}

int ensure_workspace(gnn_ctx* c, int64_t N, int64_t E) {
  if (N <= c->cap_nodes && E <= c->cap_edges) return GNN_OK;
  const int64_t n = N > c->cap_nodes ? N : c->cap_nodes;
  const int64_t e = E > c->cap_edges ? E : c->cap_edges;
  const int64_t H = c->cfg.hidden;
  const int64_t rs_tiles = (e + kRadixTile - 1) / kRadixTile;
  auto al = [](int64_t b) { return (b + 255) & ~int64_t(255); };
  const int64_t sz_e_int = al(4 * (e > 0 ? e : 1));
  // edge and node state use the row-tiled layout: rows padded to whole 128-row tiles
  const int64_t e_pad = (e + kTileRows - 1) / kTileRows * kTileRows;
  const int64_t n_pad = (n + kTileRows - 1) / kTileRows * kTileRows;
  const int64_t se = state_bytes(c);                   // stored-state element: fp32 or bf16
  const int64_t total = 8 * sz_e_int + al(4 * 256 * (rs_tiles > 0 ? rs_tiles : 1)) + al(4 * (n + 1)) +
                        al(se * e_pad * H) + 2 * al(se * n_pad * H) + 2 * al(4 * n * H);
  free_workspace(c);
  void* ws = nullptr;
  cudaError_t err = dev_alloc(&ws, (size_t)total);
  if (err != cudaSuccess) return cuda_fail(err);
  c->ws = ws;
  uint8_t* q = (uint8_t*)ws;
  auto take = [&](int64_t bytes) { uint8_t* r = q; q += al(bytes); return r; };
  c->keys_a = (int*)take(4 * e); c->keys_b = (int*)take(4 * e);
  c->vals_a = (int*)take(4 * e); c->vals_b = (int*)take(4 * e);
  c->src_c = (int*)take(4 * e); c->perm = (int*)take(4 * e);
  c->src_sorted = (int*)take(4 * e); c->dst_sorted = (int*)take(4 * e);
  c->hist = (int*)take(4 * 256 * (rs_tiles > 0 ? rs_tiles : 1));
  c->rowptr = (int*)take(4 * (n + 1));
  c->e = take(se * e_pad * H);
  c->h = take(se * n_pad * H);
  c->agg = take(se * n_pad * H);
  c->ps = (float*)take(4 * n * H);
  c->pd = (float*)take(4 * n * H);
  c->cap_nodes = n;
  c->cap_edges = e;
  return GNN_OK;
}

int build_csr(gnn_ctx* c, const int32_t* ei, int N, int E, cudaStream_t st) {
  const int tb = 256;
  int n_bits = 0;
  while (n_bits < 31 && (N >> n_bits) != 0) ++n_bits;
  const int n_passes = ((n_bits > 0 ? n_bits : 1) + 7) / 8;
  const int pr = prof_begin(c, 0, 3 + 3 * n_passes, st);
  cudaError_t le = cudaSuccess;                        // first launch error
  auto chk = [&](cudaError_t e) { if (le == cudaSuccess) le = e; };
  chk(launch_pdl(csr_keys_kernel, blocks_for(E, tb), tb, 0, st, ei, E, N, c->keys_a, c->vals_a, c->src_c, c->d_err));
  int bits = 0;
  while (bits < 31 && (N >> bits) != 0) ++bits;        // keys lie in [0, N]
  if (bits == 0) bits = 1;
  const int passes = (bits + 7) / 8;
  const int tiles = (int)blocks_for(E, kRadixTile);
  int *kin = c->keys_a, *vin = c->vals_a, *kout = c->keys_b, *vout = c->vals_b;
  for (int ps = 0; ps < passes; ++ps) {
    const int shift = 8 * ps;
    chk(launch_pdl(radix_count_kernel, tiles, kRadixThreads, 0, st, (const int*)kin, E, shift, tiles, c->hist));
    chk(launch_pdl(radix_offsets_kernel, 1, kOffsetsThreads, 0, st, c->hist, tiles));
    chk(launch_pdl(radix_scatter_kernel, tiles, kRadixThreads, 0, st, (const int*)kin, (const int*)vin, kout, vout, E,
                   shift, tiles, (const int*)c->hist));
    int* t = kin; kin = kout; kout = t;
    t = vin; vin = vout; vout = t;
  }
  c->key_sorted = kin;
  chk(launch_pdl(csr_gather_kernel, blocks_for(E, tb), tb, 0, st, (const int*)kin, (const int*)vin,
                 (const int*)c->src_c, E, N, c->perm, c->src_sorted, c->dst_sorted));
  chk(launch_pdl(csr_rowptr_kernel, blocks_for((int64_t)N + 1, tb), tb, 0, st, (const int*)kin, E, N, c->rowptr));
  prof_end(c, pr, st);
  const cudaError_t err = le != cudaSuccess ? le : cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

}  // namespace

extern "C" {

const char* gnn_error_string(int code) {
  switch (code) {
    case GNN_OK: return "ok";
    case GNN_ERR_INVALID_ARG: return "invalid argument";
    case GNN_ERR_BAD_WEIGHTS: return "bad weight blob";
    case GNN_ERR_OOM: return "device out of memory";
    case GNN_ERR_CUDA: return "CUDA error";
    case GNN_ERR_INDEX_RANGE: return "edge endpoint out of range";
    case GNN_ERR_DEVICE_TIMEOUT: return "device pipeline wait timed out";
    case GNN_ERR_CAPACITY: return "output buffer too small";
    default: return "unknown status";
  }
}

int gnn_create(const gnn_config* cfg, const void* weights_host, size_t weights_bytes, gnn_ctx** out) {
  if (!cfg || !weights_host || !out) return GNN_ERR_INVALID_ARG;
  *out = nullptr;
  const int H = cfg->hidden, L = cfg->mlp_layers, Fn = cfg->n_node_feat;
  if (cfg->version != 1 || (H != 64 && H != 128) || L < 2 || L > 4 || Fn < 2 || Fn > 16 ||
      cfg->n_edge_feat != 2 || cfg->n_iters < 0 || cfg->n_iters > 64 ||
      (cfg->precision != GNN_PRECISION_FP32 && cfg->precision != GNN_PRECISION_BF16) || !(cfg->ln_eps > 0.f))
    return GNN_ERR_INVALID_ARG;
  if (weights_bytes < (size_t)kHeaderBytes) return GNN_ERR_BAD_WEIGHTS;
  const uint8_t* blob = (const uint8_t*)weights_host;
  int32_t hdr[8];
  float eps;
  int64_t n_floats;
  std::memcpy(hdr, blob, 32);
  std::memcpy(&eps, blob + 32, 4);
  std::memcpy(&n_floats, blob + 40, 8);
  if ((uint32_t)hdr[0] != kBlobMagic || hdr[1] != 1 || hdr[2] != Fn || hdr[3] != 2 || hdr[4] != H ||
      hdr[5] != cfg->n_iters || hdr[6] != L || hdr[7] != cfg->precision || eps != cfg->ln_eps)
    return GNN_ERR_BAD_WEIGHTS;
  const int in1[N_MLP] = {Fn, 2, 3 * H, 2 * H, 3 * H};
  int64_t want = H + 1;
  for (int m = 0; m < N_MLP; ++m) want += (int64_t)H * in1[m] + 3 * H + (int64_t)(L - 1) * (H * H + 3 * H);
  if (n_floats != want || weights_bytes != (size_t)kHeaderBytes + 4 * (size_t)want) return GNN_ERR_BAD_WEIGHTS;

  // locate arrays
  const float* f = (const float*)(blob + kHeaderBytes);
  Layer lay[N_MLP][4];
  for (int m = 0; m < N_MLP; ++m)
    for (int l = 0; l < L; ++l) {
      const int in = l == 0 ? in1[m] : H;
      lay[m][l] = {f, f + (size_t)H * in, f + (size_t)H * in + H, f + (size_t)H * in + 2 * H, in};
      f += (size_t)H * in + 3 * H;
    }
  const float* head_w = f;
  const float* head_b = f + H;

  // Every Linear layer here feeds a LayerNorm, whose first step subtracts the
  // mean over the H outputs.  That subtraction is linear, so it is folded into
  // the layer: each weight column and the bias are centred over the output
  // rows (W' = (I - 11^T/H) W, b' = b - mean(b)).  The kernels then receive
  // zero-mean pre-activations and compute only the variance.  Centred copies
  // are kept in `centred` and the Layer pointers redirected to them.
  // The bf16 model keeps its weights as given (bf16 values): centring would take them off the
  // bf16 grid, so its kernels subtract the LayerNorm mean themselves.
  const bool bf = cfg->precision == GNN_PRECISION_BF16;
  std::vector<std::vector<float>> centred;
  centred.reserve(2 * N_MLP * L);
  for (int m = 0; m < N_MLP && !bf; ++m)
    for (int l = 0; l < L; ++l) {
      Layer& ly = lay[m][l];
      std::vector<float> Wc, bc;
      centre_layer(ly.W, ly.b, H, ly.in, Wc, bc);
      centred.push_back(std::move(Wc));
      ly.W = centred.back().data();
      centred.push_back(std::move(bc));
      ly.b = centred.back().data();
    }

  gnn_ctx* c = new (std::nothrow) gnn_ctx();
  if (!c) return GNN_ERR_OOM;
  c->cfg = *cfg;
  cudaError_t err = cudaGetDevice(&c->device);
  if (err == cudaSuccess) err = cudaDeviceGetAttribute(&c->n_sm, cudaDevAttrMultiProcessorCount, c->device);
  if (err == cudaSuccess)
    err = bf ? ((H == 128) ? set_all_attrs<128, true>() : set_all_attrs<64, true>())
             : ((H == 128) ? set_all_attrs<128, false>() : set_all_attrs<64, false>());
  if (err != cudaSuccess) { delete c; return cuda_fail(err); }

  // matrices
  std::vector<std::pair<const Layer*, int>> mats;   // (layer, column offset)
  auto add_mat = [&](const Layer* ly, int col0) { mats.push_back({ly, col0}); return (int)mats.size() - 1; };
  const int en_s = add_mat(&lay[EDGE_NET][0], 0), en_d = add_mat(&lay[EDGE_NET][0], H),
            en_e = add_mat(&lay[EDGE_NET][0], 2 * H);
  const int cl_s = add_mat(&lay[CLASSIFIER][0], 0), cl_d = add_mat(&lay[CLASSIFIER][0], H),
            cl_e = add_mat(&lay[CLASSIFIER][0], 2 * H);
  const int nn_h = add_mat(&lay[NODE_NET][0], 0), nn_a = add_mat(&lay[NODE_NET][0], H);
  int deep[N_MLP][4];
  for (int m = 0; m < N_MLP; ++m)
    for (int l = 1; l < L; ++l) deep[m][l] = add_mat(&lay[m][l], 0);
  c->mat_bytes = (bf ? 1u : 2u) * H * H * 2u;
  std::vector<uint8_t> packed((size_t)c->mat_bytes * mats.size());
  for (size_t i = 0; i < mats.size(); ++i)
    pack_block(mats[i].first->W, mats[i].first->in, mats[i].second, H, !bf, packed.data() + i * c->mat_bytes);

  // kernel plans
  auto jobs = [](KernelPlan& pl, std::initializer_list<int> ids, int acc_mask = 0) {
    pl.n_jobs = 0;
    for (int id : ids) { pl.job_acc[pl.n_jobs] = (acc_mask >> pl.n_jobs) & 1; pl.job_mat[pl.n_jobs++] = id; }
  };
  auto add_deep = [&](KernelPlan& pl, int m) {
    for (int l = 1; l < L; ++l) { pl.job_acc[pl.n_jobs] = 0; pl.job_mat[pl.n_jobs++] = deep[m][l]; }
  };
  auto bgb = [&](std::vector<float>& v, int m, int l0) {
    for (int l = l0; l < L; ++l) { push(v, lay[m][l].b, H); push(v, lay[m][l].g, H); push(v, lay[m][l].be, H); }
  };
  for (int target = 0; target < 2; ++target) {           // node encoder -> edge net / classifier
    KernelPlan& pl = c->plan[target];
    pl.n_jobs = 0;
    add_deep(pl, NODE_ENC);
    pl.job_mat[pl.n_jobs++] = target == 0 ? en_s : cl_s;
    pl.job_mat[pl.n_jobs++] = target == 0 ? en_d : cl_d;
    for (int k = 0; k < Fn; ++k)                        // first-layer weight, transposed
      for (int i = 0; i < H; ++i) pl.vecs.push_back(lay[NODE_ENC][0].W[(size_t)i * Fn + k]);
    bgb(pl.vecs, NODE_ENC, 0);
    push(pl.vecs, lay[target == 0 ? EDGE_NET : CLASSIFIER][0].b, H);
  }
  {  // edge encoder
    KernelPlan& pl = c->plan[2];
    pl.n_jobs = 0;
    add_deep(pl, EDGE_ENC);
    for (int k = 0; k < 2; ++k)
      for (int i = 0; i < H; ++i) pl.vecs.push_back(lay[EDGE_ENC][0].W[(size_t)i * 2 + k]);
    bgb(pl.vecs, EDGE_ENC, 0);
  }
  {  // edge update
    KernelPlan& pl = c->plan[3];
    jobs(pl, {en_e});
    add_deep(pl, EDGE_NET);
    push(pl.vecs, lay[EDGE_NET][0].g, H);
    push(pl.vecs, lay[EDGE_NET][0].be, H);
    bgb(pl.vecs, EDGE_NET, 1);
  }
  for (int target = 0; target < 2; ++target) {           // node update -> edge net / classifier
    KernelPlan& pl = c->plan[4 + target];
    jobs(pl, {nn_h, nn_a}, 0b10);
    add_deep(pl, NODE_NET);
    pl.job_acc[pl.n_jobs] = 0; pl.job_mat[pl.n_jobs++] = target == 0 ? en_s : cl_s;
    pl.job_acc[pl.n_jobs] = 0; pl.job_mat[pl.n_jobs++] = target == 0 ? en_d : cl_d;
    bgb(pl.vecs, NODE_NET, 0);
    push(pl.vecs, lay[target == 0 ? EDGE_NET : CLASSIFIER][0].b, H);
  }
  {  // classifier
    KernelPlan& pl = c->plan[6];
    jobs(pl, {cl_e});
    add_deep(pl, CLASSIFIER);
    push(pl.vecs, lay[CLASSIFIER][0].g, H);
    push(pl.vecs, lay[CLASSIFIER][0].be, H);
    bgb(pl.vecs, CLASSIFIER, 1);
    push(pl.vecs, head_w, H);
    push(pl.vecs, head_b, 1);
  }

  for (int i = 0; i < 7; ++i) finish_vecs(c->plan[i].vecs, H);
  err = dev_alloc((void**)&c->d_mats, packed.size());
  if (err == cudaSuccess) err = cudaMemcpy(c->d_mats, packed.data(), packed.size(), cudaMemcpyHostToDevice);
  for (int i = 0; i < 7 && err == cudaSuccess; ++i) {
    err = dev_alloc((void**)&c->plan[i].d_vecs, c->plan[i].vecs.size() * 4);
    if (err == cudaSuccess)
      err = cudaMemcpy(c->plan[i].d_vecs, c->plan[i].vecs.data(), c->plan[i].vecs.size() * 4, cudaMemcpyHostToDevice);
  }
#ifdef GNN_TRACE
  if (err == cudaSuccess) err = cudaMalloc(&c->trace, 3 * kTraceEvents * 8);
  if (err == cudaSuccess) err = cudaMemset(c->trace, 0, 3 * kTraceEvents * 8);
  if (const char* k = getenv("GNN_TRACE_KIND")) c->trace_kind = atoi(k);
#endif
  if (err == cudaSuccess) err = dev_alloc((void**)&c->d_err, 4);
  if (err == cudaSuccess) err = cudaMemset(c->d_err, 0, 4);
  if (err != cudaSuccess) { gnn_destroy(c); return cuda_fail(err); }
  *out = c;
  return GNN_OK;
}

int gnn_reserve(gnn_ctx* ctx, int64_t max_nodes, int64_t max_edges) {
  if (!count_ok(max_nodes) || !count_ok(max_edges) || !ctx) return GNN_ERR_INVALID_ARG;
  return ensure_workspace(ctx, max_nodes, max_edges);
}

int gnn_infer(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
              int64_t n_edges, float* edge_scores, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !count_ok(n_edges) || !ctx) return GNN_ERR_INVALID_ARG;
  if (n_edges == 0) return GNN_OK;
  if (n_nodes == 0 || !node_feats || !edge_index || !edge_scores) return GNN_ERR_INVALID_ARG;
  int rc = ensure_workspace(ctx, n_nodes, n_edges);
  if (rc != GNN_OK) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const int N = (int)n_nodes, E = (int)n_edges;
  rc = build_csr(ctx, edge_index, N, E, st);
  if (rc != GNN_OK) return rc;
  ctx->last_nodes = N;
  ctx->last_edges = E;
  const bool bf = ctx->cfg.precision == GNN_PRECISION_BF16;
  if (ctx->cfg.hidden == 128)
    return bf ? run_network<128, true>(ctx, node_feats, N, E, edge_scores, st)
              : run_network<128, false>(ctx, node_feats, N, E, edge_scores, st);
  return bf ? run_network<64, true>(ctx, node_feats, N, E, edge_scores, st)
            : run_network<64, false>(ctx, node_feats, N, E, edge_scores, st);
}

int gnn_infer_host(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
                   int64_t n_edges, float* edge_scores, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !count_ok(n_edges) || !ctx) return GNN_ERR_INVALID_ARG;
  if (n_edges == 0) return GNN_OK;
  if (n_nodes == 0 || !node_feats || !edge_index || !edge_scores) return GNN_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  const size_t bx = (size_t)n_nodes * ctx->cfg.n_node_feat * 4, be = (size_t)n_edges * 8,
               bs = (size_t)n_edges * 4;
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  const size_t need = al(bx) + al(be) + al(bs);
  if (need > ctx->stage_bytes) {
    if (ctx->stage) { cudaStreamSynchronize(st); cudaFree(ctx->stage); ctx->stage = nullptr; ctx->stage_bytes = 0; }
    const cudaError_t err = dev_alloc(&ctx->stage, need);
    if (err != cudaSuccess) return cuda_fail(err);
    ctx->stage_bytes = need;
  }
  uint8_t* q = (uint8_t*)ctx->stage;
  float* dx = (float*)q;
  int32_t* de = (int32_t*)(q + al(bx));
  float* ds = (float*)(q + al(bx) + al(be));
  int pr = prof_begin(ctx, 6, 2, st);
  cudaError_t err = cudaMemcpyAsync(dx, node_feats, bx, cudaMemcpyHostToDevice, st);
  if (err == cudaSuccess) err = cudaMemcpyAsync(de, edge_index, be, cudaMemcpyHostToDevice, st);
  prof_end(ctx, pr, st);
  if (err != cudaSuccess) return cuda_fail(err);
  int rc = gnn_infer(ctx, dx, de, n_nodes, n_edges, ds, stream);
  if (rc != GNN_OK) return rc;
  pr = prof_begin(ctx, 6, 1, st);
  err = cudaMemcpyAsync(edge_scores, ds, bs, cudaMemcpyDeviceToHost, st);
  prof_end(ctx, pr, st);
  if (err != cudaSuccess) return cuda_fail(err);
  return gnn_status(ctx, stream);
}

int gnn_filter_load(gnn_ctx* ctx, const void* weights_host, size_t weights_bytes) {
  if (!ctx || !weights_host) return GNN_ERR_INVALID_ARG;
  const int H = ctx->cfg.hidden, Fn = ctx->cfg.n_node_feat;
  const bool bf = ctx->cfg.precision == GNN_PRECISION_BF16;
  if (weights_bytes < (size_t)kHeaderBytes) return GNN_ERR_BAD_WEIGHTS;
  const uint8_t* blob = (const uint8_t*)weights_host;
  int32_t hdr[8];
  float eps;
  int64_t n_floats;
  std::memcpy(hdr, blob, 32);
  std::memcpy(&eps, blob + 32, 4);
  std::memcpy(&n_floats, blob + 40, 8);
  const int L = hdr[4];
  if ((uint32_t)hdr[0] != kFilterMagic || hdr[1] != 1 || hdr[2] != Fn || hdr[3] != H || L < 2 || L > 4 ||
      hdr[5] != ctx->cfg.precision || !(eps > 0.f))
    return GNN_ERR_BAD_WEIGHTS;
  const int64_t want = (int64_t)H * 2 * Fn + 3 * H + (int64_t)(L - 1) * (H * H + 3 * H) + H + 1;
  if (n_floats != want || weights_bytes != (size_t)kHeaderBytes + 4 * (size_t)want) return GNN_ERR_BAD_WEIGHTS;
  const float* f = (const float*)(blob + kHeaderBytes);
  std::vector<Layer> lay(L);
  for (int l = 0; l < L; ++l) {
    const int in = l == 0 ? 2 * Fn : H;
    lay[l] = {f, f + (size_t)H * in, f + (size_t)H * in + H, f + (size_t)H * in + 2 * H, in};
    f += (size_t)H * in + 3 * H;
  }
  const float* head = f;
  std::vector<std::vector<float>> centred(2 * L);
  if (!bf)
    for (int l = 0; l < L; ++l) {
      centre_layer(lay[l].W, lay[l].b, H, lay[l].in, centred[2 * l], centred[2 * l + 1]);
      lay[l].W = centred[2 * l].data();
      lay[l].b = centred[2 * l + 1].data();
    }
  KernelPlan pl;
  for (int l = 1; l < L; ++l) { pl.job_acc[pl.n_jobs] = 0; pl.job_mat[pl.n_jobs] = l - 1; ++pl.n_jobs; }
  for (int k = 0; k < 2 * Fn; ++k)                   // first-layer weight, transposed
    for (int i = 0; i < H; ++i) pl.vecs.push_back(lay[0].W[(size_t)i * 2 * Fn + k]);
  for (int l = 0; l < L; ++l) { push(pl.vecs, lay[l].b, H); push(pl.vecs, lay[l].g, H); push(pl.vecs, lay[l].be, H); }
  push(pl.vecs, head, H + 1);
  finish_vecs(pl.vecs, H);
  std::vector<uint8_t> packed((size_t)ctx->mat_bytes * (L - 1));
  for (int l = 1; l < L; ++l) pack_block(lay[l].W, H, 0, H, !bf, packed.data() + (size_t)(l - 1) * ctx->mat_bytes);
  // replace a previous filter
  if (ctx->filter_plan.d_vecs) { cudaFree(ctx->filter_plan.d_vecs); ctx->filter_plan.d_vecs = nullptr; }
  if (ctx->d_filter_mats) { cudaFree(ctx->d_filter_mats); ctx->d_filter_mats = nullptr; }
  ctx->filter_layers = 0;
  cudaError_t err = dev_alloc((void**)&ctx->d_filter_mats, packed.size());
  if (err == cudaSuccess) err = cudaMemcpy(ctx->d_filter_mats, packed.data(), packed.size(), cudaMemcpyHostToDevice);
  if (err == cudaSuccess) err = dev_alloc((void**)&pl.d_vecs, pl.vecs.size() * 4);
  if (err == cudaSuccess) err = cudaMemcpy(pl.d_vecs, pl.vecs.data(), pl.vecs.size() * 4, cudaMemcpyHostToDevice);
  if (err != cudaSuccess) {
    if (pl.d_vecs) cudaFree(pl.d_vecs);
    if (ctx->d_filter_mats) { cudaFree(ctx->d_filter_mats); ctx->d_filter_mats = nullptr; }
    return cuda_fail(err);
  }
  pl.wmats = ctx->d_filter_mats;
  ctx->filter_plan = std::move(pl);
  ctx->filter_layers = L;
  ctx->filter_eps = eps;
  return GNN_OK;
}

int gnn_filter_edges(gnn_ctx* ctx, const float* node_feats, const int32_t* edge_index, int64_t n_nodes,
                     int64_t n_edges, float threshold, float* edge_scores, int32_t* kept_index, int32_t* kept_id,
                     int32_t* n_kept, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !count_ok(n_edges) || !ctx || !n_kept) return GNN_ERR_INVALID_ARG;
  if (ctx->filter_layers == 0) return GNN_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  if (n_edges == 0) {
    const cudaError_t err = cudaMemsetAsync(n_kept, 0, sizeof(int32_t), st);
    return err == cudaSuccess ? GNN_OK : cuda_fail(err);
  }
  if (n_nodes == 0 || !node_feats || !edge_index || !edge_scores || !kept_index) return GNN_ERR_INVALID_ARG;
  int rc = ensure_workspace(ctx, n_nodes, n_edges);          // block counts live in the sort keys' buffer
  if (rc != GNN_OK) return rc;
  const int N = (int)n_nodes, E = (int)n_edges;
  TileParams p{};
  p.n_rows = E;
  p.n_nodes = N;
  p.n_layers = ctx->filter_layers;
  p.n_feat = ctx->cfg.n_node_feat;
  p.eps = ctx->filter_eps;
  p.x = node_feats;
  p.x_stride = ctx->cfg.n_node_feat;
  p.ei_in = edge_index;
  p.scores = edge_scores;
  p.err = ctx->d_err;
  const bool bf = ctx->cfg.precision == GNN_PRECISION_BF16;
  if (ctx->cfg.hidden == 128) {
    if (bf) launch_tile<TileKind::Filter, 128, true>(ctx, ctx->filter_plan, p, st);
    else launch_tile<TileKind::Filter, 128, false>(ctx, ctx->filter_plan, p, st);
  } else {
    if (bf) launch_tile<TileKind::Filter, 64, true>(ctx, ctx->filter_plan, p, st);
    else launch_tile<TileKind::Filter, 64, false>(ctx, ctx->filter_plan, p, st);
  }
  const int nb = (int)blocks_for(E, kCompactBlock);
  int* counts = ctx->keys_a;
  compact_count_kernel<<<nb, kCompactThreads, 0, st>>>(edge_scores, E, threshold, counts);
  compact_scan_kernel<<<1, 1024, 0, st>>>(counts, nb, n_kept);
  compact_scatter_kernel<<<nb, kCompactThreads, 0, st>>>(edge_scores, edge_index, E, threshold, counts, n_kept,
                                                          kept_index, kept_id);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

int gnn_embed_load(gnn_ctx* ctx, const void* weights_host, size_t weights_bytes) {
  if (!ctx || !weights_host) return GNN_ERR_INVALID_ARG;
  const int H = ctx->cfg.hidden, Fn = ctx->cfg.n_node_feat;
  const bool bf = ctx->cfg.precision == GNN_PRECISION_BF16;
  if (weights_bytes < (size_t)kHeaderBytes) return GNN_ERR_BAD_WEIGHTS;
  const uint8_t* blob = (const uint8_t*)weights_host;
  int32_t hdr[8];
  float eps;
  int64_t n_floats;
  std::memcpy(hdr, blob, 32);
  std::memcpy(&eps, blob + 32, 4);
  std::memcpy(&n_floats, blob + 40, 8);
  const int L = hdr[4], D = hdr[6];
  if ((uint32_t)hdr[0] != kEmbedMagic || hdr[1] != 1 || hdr[2] != Fn || hdr[3] != H || L < 2 || L > 4 ||
      hdr[5] != ctx->cfg.precision || D < 1 || D > kMaxEmbedDim || !(eps > 0.f))
    return GNN_ERR_BAD_WEIGHTS;
  const int64_t want = (int64_t)H * Fn + 3 * H + (int64_t)(L - 1) * (H * H + 3 * H) + (int64_t)D * H + D;
  if (n_floats != want || weights_bytes != (size_t)kHeaderBytes + 4 * (size_t)want) return GNN_ERR_BAD_WEIGHTS;
  const float* f = (const float*)(blob + kHeaderBytes);
  std::vector<Layer> lay(L);
  for (int l = 0; l < L; ++l) {
    const int in = l == 0 ? Fn : H;
    lay[l] = {f, f + (size_t)H * in, f + (size_t)H * in + H, f + (size_t)H * in + 2 * H, in};
    f += (size_t)H * in + 3 * H;
  }
  const float* wout = f;                                  // [D, H] then b_out [D]
  std::vector<std::vector<float>> centred(2 * L);
  if (!bf)
    for (int l = 0; l < L; ++l) {
      centre_layer(lay[l].W, lay[l].b, H, lay[l].in, centred[2 * l], centred[2 * l + 1]);
      lay[l].W = centred[2 * l].data();
      lay[l].b = centred[2 * l + 1].data();
    }
  KernelPlan pl;
  for (int l = 1; l < L; ++l) { pl.job_acc[pl.n_jobs] = 0; pl.job_mat[pl.n_jobs] = l - 1; ++pl.n_jobs; }
  for (int k = 0; k < Fn; ++k)                        // first-layer weight, transposed
    for (int i = 0; i < H; ++i) pl.vecs.push_back(lay[0].W[(size_t)i * Fn + k]);
  for (int l = 0; l < L; ++l) { push(pl.vecs, lay[l].b, H); push(pl.vecs, lay[l].g, H); push(pl.vecs, lay[l].be, H); }
  push(pl.vecs, wout, (size_t)D * H + D);
  finish_vecs(pl.vecs, H);
  std::vector<uint8_t> packed((size_t)ctx->mat_bytes * (L - 1));
  for (int l = 1; l < L; ++l) pack_block(lay[l].W, H, 0, H, !bf, packed.data() + (size_t)(l - 1) * ctx->mat_bytes);
  if (ctx->embed_plan.d_vecs) { cudaFree(ctx->embed_plan.d_vecs); ctx->embed_plan.d_vecs = nullptr; }
  if (ctx->d_embed_mats) { cudaFree(ctx->d_embed_mats); ctx->d_embed_mats = nullptr; }
  ctx->embed_layers = 0;
  cudaError_t err = dev_alloc((void**)&ctx->d_embed_mats, packed.size());
  if (err == cudaSuccess) err = cudaMemcpy(ctx->d_embed_mats, packed.data(), packed.size(), cudaMemcpyHostToDevice);
  if (err == cudaSuccess) err = dev_alloc((void**)&pl.d_vecs, pl.vecs.size() * 4);
  if (err == cudaSuccess) err = cudaMemcpy(pl.d_vecs, pl.vecs.data(), pl.vecs.size() * 4, cudaMemcpyHostToDevice);
  if (err != cudaSuccess) {
    if (pl.d_vecs) cudaFree(pl.d_vecs);
    if (ctx->d_embed_mats) { cudaFree(ctx->d_embed_mats); ctx->d_embed_mats = nullptr; }
    return cuda_fail(err);
  }
  pl.wmats = ctx->d_embed_mats;
  ctx->embed_plan = std::move(pl);
  ctx->embed_layers = L;
  ctx->embed_dim = D;
  ctx->embed_eps = eps;
  return GNN_OK;
}

int gnn_embed(gnn_ctx* ctx, const float* node_feats, int64_t n_nodes, float* embedding, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !ctx || ctx->embed_layers == 0) return GNN_ERR_INVALID_ARG;
  if (n_nodes == 0) return GNN_OK;
  if (!node_feats || !embedding) return GNN_ERR_INVALID_ARG;
  TileParams p{};
  p.n_rows = (int)n_nodes;
  p.n_nodes = (int)n_nodes;
  p.n_layers = ctx->embed_layers;
  p.n_feat = ctx->cfg.n_node_feat;
  p.eps = ctx->embed_eps;
  p.x = node_feats;
  p.x_stride = ctx->cfg.n_node_feat;
  p.emb = embedding;
  p.emb_dim = ctx->embed_dim;
  p.err = ctx->d_err;
  cudaStream_t st = (cudaStream_t)stream;
  const bool bf = ctx->cfg.precision == GNN_PRECISION_BF16;
  if (ctx->cfg.hidden == 128) {
    if (bf) launch_tile<TileKind::Embed, 128, true>(ctx, ctx->embed_plan, p, st);
    else launch_tile<TileKind::Embed, 128, false>(ctx, ctx->embed_plan, p, st);
  } else {
    if (bf) launch_tile<TileKind::Embed, 64, true>(ctx, ctx->embed_plan, p, st);
    else launch_tile<TileKind::Embed, 64, false>(ctx, ctx->embed_plan, p, st);
  }
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

int gnn_build_graph(gnn_ctx* ctx, const float* embedding, int emb_dim, const float* node_feats, int64_t n_nodes,
                    float radius, int64_t max_edges, int32_t* edge_index, int32_t* n_edges, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !count_ok(max_edges) || !ctx || emb_dim < 1 || emb_dim > kMaxEmbedDim ||
      !(radius > 0.f) || !n_edges)
    return GNN_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  if (n_nodes == 0) {
    const cudaError_t err = cudaMemsetAsync(n_edges, 0, sizeof(int32_t), st);
    return err == cudaSuccess ? GNN_OK : cuda_fail(err);
  }
  if (!embedding || !node_feats || (max_edges > 0 && !edge_index)) return GNN_ERR_INVALID_ARG;
  const int N = (int)n_nodes, tb = 256;
  // grid over 4 embedding coordinates when there are at least 4 (on the full event's 8-dimensional
  // embedding, when the writing pass still searched again: 9.0 ms against 14.8 ms with 3), else over 3
  const int K = emb_dim >= 4 ? 4 : 3;
  const int grid = frnn_grid(radius, K);
  int n_cells = 1;
  for (int k = 0; k < K; ++k) n_cells *= grid;
  const int tiles = (int)blocks_for(N, kRadixTile);
  const int chunks = (emb_dim + 3) / 4;                   // float4 chunks per sorted embedding
  // partner chains kept by the counting pass: one first chunk per hit, pool chunks after them (a hit
  // whose chain cannot grow is searched again by the writing pass)
  const int64_t pool64 = ctx->graph_pool >= 0 ? ctx->graph_pool : (int64_t)N;
  const int pool = (int)(pool64 < (int64_t)INT_MAX - N ? pool64 : (int64_t)INT_MAX - N);
  // scratch: emb_s [N, 4 * chunks] (first, 16-byte aligned), partner chunks, r_s, keys/vals (two
  // buffers each), per-hit counts, per-block sums, radix histograms, cell starts, the pool counter
  const int nb = (int)blocks_for(N, tb);
  const size_t chain_ints = ((size_t)N + (size_t)pool) * kFrnnChunk;
  const size_t need = 4 * (size_t)chunks * N + chain_ints + 6 * (size_t)N + (size_t)nb + 256 * (size_t)tiles +
                      (size_t)n_cells + 2;
  if (need > ctx->aux_ints) {
    if (ctx->aux) { cudaStreamSynchronize(st); cudaFree(ctx->aux); ctx->aux = nullptr; ctx->aux_ints = 0; }
    const cudaError_t err = dev_alloc((void**)&ctx->aux, need * sizeof(int));
    if (err != cudaSuccess) return cuda_fail(err);
    ctx->aux_ints = need;
  }
  float4* emb_s = (float4*)ctx->aux;
  int* chains = (int*)(ctx->aux + 4 * (size_t)chunks * N);
  float* r_s = (float*)(chains + chain_ints);
  int* keys_a = (int*)(r_s + N);
  int* keys_b = keys_a + N;
  int* vals_a = keys_b + N;
  int* vals_b = vals_a + N;
  int* counts = vals_b + N;
  int* block_sums = counts + N;
  int* hist = block_sums + nb;
  int* cell_start = hist + 256 * (size_t)tiles;
  int* next_chunk = cell_start + n_cells + 1;
  if (K == 4) frnn_cell_kernel<4><<<nb, tb, 0, st>>>(embedding, N, emb_dim, grid, keys_a, vals_a);
  else frnn_cell_kernel<3><<<nb, tb, 0, st>>>(embedding, N, emb_dim, grid, keys_a, vals_a);
  int bits = 0;
  while (bits < 31 && ((n_cells - 1) >> bits) != 0) ++bits;
  const int passes = ((bits > 0 ? bits : 1) + 7) / 8;
  int *kin = keys_a, *vin = vals_a, *kout = keys_b, *vout = vals_b;
  for (int ps = 0; ps < passes; ++ps) {
    radix_count_kernel<<<tiles, kRadixThreads, 0, st>>>(kin, N, 8 * ps, tiles, hist);
    radix_offsets_kernel<<<1, kOffsetsThreads, 0, st>>>(hist, tiles);
    radix_scatter_kernel<<<tiles, kRadixThreads, 0, st>>>(kin, vin, kout, vout, N, 8 * ps, tiles, hist);
    int* t = kin; kin = kout; kout = t;
    t = vin; vin = vout; vout = t;
  }
  csr_rowptr_kernel<<<blocks_for((int64_t)n_cells + 1, tb), tb, 0, st>>>(kin, N, n_cells, cell_start);
  {
    const cudaError_t e0 = cudaMemsetAsync(next_chunk, 0, sizeof(int), st);
    if (e0 != cudaSuccess) return cuda_fail(e0);
  }
  const float r2 = radius * radius;
  const int xs = ctx->cfg.n_node_feat;
  const int sb = (int)blocks_for(N, kScanBlock);
  const int pb = (int)blocks_for(N, kFrnnPairsThreads);
  switch (chunks * 8 + K) {
#define GNN_FRNN_CASE(CH, KK)                                                                                    \
  case CH * 8 + KK:                                                                                              \
    frnn_gather_kernel<CH><<<nb, tb, 0, st>>>(embedding, node_feats, xs, N, emb_dim, vin, emb_s, r_s);         \
    frnn_pairs_kernel<CH, KK><<<pb, kFrnnPairsThreads, 0, st>>>(emb_s, r_s, N, r2, grid, kin, vin, cell_start, \
                                                                0, counts, nullptr, 0, nullptr, chains,          \
                                                                next_chunk, pool, ctx->d_err);                   \
    scan_reduce_kernel<<<sb, kScanBlock, 0, st>>>(counts, N, block_sums);                                      \
    compact_scan_kernel<<<1, 1024, 0, st>>>(block_sums, sb, n_edges);                                            \
    scan_apply_kernel<<<sb, kScanBlock, 0, st>>>(counts, N, block_sums);                                       \
    frnn_pairs_kernel<CH, KK><<<pb, kFrnnPairsThreads, 0, st>>>(emb_s, r_s, N, r2, grid, kin, vin, cell_start, \
                                                                1, counts, n_edges, (int)max_edges, edge_index,  \
                                                                chains, next_chunk, pool, ctx->d_err);           \
    frnn_copy_kernel<<<nb, tb, 0, st>>>(r_s, N, vin, counts, n_edges, (int)max_edges, chains, edge_index);      \
    break;
    GNN_FRNN_CASE(1, 3)
    GNN_FRNN_CASE(2, 3)
    GNN_FRNN_CASE(3, 3)
    GNN_FRNN_CASE(4, 3)
    GNN_FRNN_CASE(1, 4)
    GNN_FRNN_CASE(2, 4)
    GNN_FRNN_CASE(3, 4)
    GNN_FRNN_CASE(4, 4)
#undef GNN_FRNN_CASE
  }
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

int gnn_track_labels(gnn_ctx* ctx, const float* edge_scores, const int32_t* edge_index, int64_t n_nodes,
                     int64_t n_edges, float threshold, int32_t* labels, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || !count_ok(n_edges) || !ctx) return GNN_ERR_INVALID_ARG;
  if (n_nodes == 0) return n_edges == 0 ? GNN_OK : GNN_ERR_INVALID_ARG;
  if (!labels || (n_edges > 0 && (!edge_scores || !edge_index))) return GNN_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  const int N = (int)n_nodes, E = (int)n_edges, tb = 256;
  cc_init_kernel<<<blocks_for(N, tb), tb, 0, st>>>(labels, N);
  if (E > 0) cc_union_kernel<<<blocks_for(E, tb), tb, 0, st>>>(edge_scores, edge_index, N, E, threshold, labels, ctx->d_err);
  cc_compress_kernel<<<blocks_for(N, tb), tb, 0, st>>>(labels, N, ctx->d_err);
  cc_flatten_kernel<<<blocks_for(N, tb), tb, 0, st>>>(labels, N, ctx->d_err);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

#ifdef GNN_TRACE
int gnn_trace_read(gnn_ctx* ctx, unsigned long long* host) {
  cudaDeviceSynchronize();
  return cudaMemcpy(host, ctx->trace, 3 * kTraceEvents * 8, cudaMemcpyDeviceToHost) == cudaSuccess ? 0 : -4;
}
#endif

int gnn_debug_fail_allocs(int n) {
  if (n < 0) return GNN_ERR_INVALID_ARG;
  g_fail_allocs.store(n);
  return GNN_OK;
}

int gnn_debug_graph_pool(gnn_ctx* ctx, int64_t chunks) {
  if (!ctx) return GNN_ERR_INVALID_ARG;
  ctx->graph_pool = chunks < 0 ? -1 : chunks;
  return GNN_OK;
}

int gnn_debug_wait_timeout(gnn_ctx* ctx, int64_t limit_ns, gnn_stream_t stream) {
  if (!ctx || limit_ns <= 0 || limit_ns > (int64_t)kWaitLimitNs) return GNN_ERR_INVALID_ARG;
  wait_timeout_kernel<<<1, 32, 0, (cudaStream_t)stream>>>((uint64_t)limit_ns, ctx->d_err);
  const cudaError_t err = cudaGetLastError();
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

int gnn_profile_enable(gnn_ctx* ctx, int on) {
  if (!ctx) return GNN_ERR_INVALID_ARG;
  ctx->prof_on = on != 0;
  return GNN_OK;
}

int gnn_profile_read(gnn_ctx* ctx, double* ms, int64_t* launches, int n_groups) {
  if (!ctx || n_groups < 0) return GNN_ERR_INVALID_ARG;
  double acc[kProfGroups] = {0};
  int64_t cnt[kProfGroups] = {0};
  for (size_t i = 0; i < ctx->prof_used; ++i) {
    gnn_ctx::ProfRec& r = ctx->prof[i];
    if (cudaEventSynchronize(r.b) != cudaSuccess) return cuda_fail(cudaGetLastError());
    float t = 0.f;
    if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return cuda_fail(cudaGetLastError());
    acc[r.group] += t;
    cnt[r.group] += r.launches;
  }
  ctx->prof_used = 0;
  for (int g = 0; g < n_groups && g < kProfGroups; ++g) {
    if (ms) ms[g] = acc[g];
    if (launches) launches[g] = cnt[g];
  }
  return kProfGroups;
}

int gnn_status(gnn_ctx* ctx, gnn_stream_t stream) {
  if (!ctx) return GNN_ERR_INVALID_ARG;
  cudaError_t err = cudaStreamSynchronize((cudaStream_t)stream);
  if (err != cudaSuccess) return cuda_fail(err);
  uint32_t word = 0;
  err = cudaMemcpy(&word, ctx->d_err, 4, cudaMemcpyDeviceToHost);
  if (err == cudaSuccess) err = cudaMemset(ctx->d_err, 0, 4);
  if (err != cudaSuccess) return cuda_fail(err);
  if (word & DEV_ERR_TIMEOUT) return GNN_ERR_DEVICE_TIMEOUT;
  if (word & DEV_ERR_CAPACITY) return GNN_ERR_CAPACITY;
  if (word & DEV_ERR_INDEX_RANGE) return GNN_ERR_INDEX_RANGE;
  return GNN_OK;
}

void gnn_destroy(gnn_ctx* ctx) {
  if (!ctx) return;
  cudaDeviceSynchronize();
  free_workspace(ctx);
  if (ctx->d_mats) cudaFree(ctx->d_mats);
  for (int i = 0; i < 7; ++i)
    if (ctx->plan[i].d_vecs) cudaFree(ctx->plan[i].d_vecs);
  if (ctx->filter_plan.d_vecs) cudaFree(ctx->filter_plan.d_vecs);
  if (ctx->d_filter_mats) cudaFree(ctx->d_filter_mats);
  if (ctx->embed_plan.d_vecs) cudaFree(ctx->embed_plan.d_vecs);
  if (ctx->d_embed_mats) cudaFree(ctx->d_embed_mats);
  if (ctx->aux) cudaFree(ctx->aux);
  if (ctx->d_err) cudaFree(ctx->d_err);
  if (ctx->stage) cudaFree(ctx->stage);
#ifdef GNN_TRACE
  if (ctx->trace) cudaFree(ctx->trace);
#endif
  for (auto& r : ctx->prof) { cudaEventDestroy(r.a); cudaEventDestroy(r.b); }
  delete ctx;
}

int gnn_debug_copy(gnn_ctx* ctx, int which, void* dst, size_t bytes, gnn_stream_t stream) {
  if (!ctx || !dst || !ctx->ws) return GNN_ERR_INVALID_ARG;
  const int64_t N = ctx->last_nodes, E = ctx->last_edges, H = ctx->cfg.hidden;
  const void* src = nullptr;
  size_t need = 0;
  switch (which) {
    case 0: src = ctx->rowptr; need = 4 * (size_t)(N + 1); break;
    case 1: src = ctx->perm; need = 4 * (size_t)E; break;
    case 2: src = ctx->src_sorted; need = 4 * (size_t)E; break;
    case 3: src = ctx->h; need = state_bytes(ctx) * (size_t)((N + kTileRows - 1) / kTileRows * kTileRows * H); break;
    case 4: src = ctx->e; need = state_bytes(ctx) * (size_t)((E + kTileRows - 1) / kTileRows * kTileRows * H); break;
    default: return GNN_ERR_INVALID_ARG;
  }
  if (bytes < need) return GNN_ERR_INVALID_ARG;
  const cudaError_t err = cudaMemcpyAsync(dst, src, need, cudaMemcpyDeviceToDevice, (cudaStream_t)stream);
  return err == cudaSuccess ? GNN_OK : cuda_fail(err);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free CSR build: the radix-sort scratch lives in one file-scope
// device array instead of context workspace.  Layout (int32 words):
// keys_a | keys_b | vals_a | vals_b | src_clamped (GNN_CSR_NOALLOC_MAX_EDGES
// each) | per-tile digit histograms (256 x 256).  Host code must not use the
// array's name as a device address: every call asks cudaGetSymbolAddress for
// it, with the caller's device current.  The address is not cached, because it
// belongs to the current context's copy of the module: it changes after
// cudaDeviceReset and differs under another context on the same device.
static_assert((GNN_CSR_NOALLOC_MAX_EDGES + kRadixTile - 1) / kRadixTile <= 256, "histogram area too small");
static __device__ __align__(256) unsigned char g_csr_noalloc_scratch[GNN_CSR_NOALLOC_SCRATCH_BYTES];

extern "C" int gnn_csr_build_noalloc(const int32_t* edge_index, int64_t n_nodes, int64_t n_edges,
                                     int32_t* rowptr, int32_t* perm, int32_t* src_sorted, gnn_stream_t stream) {
  if (!count_ok(n_nodes) || n_edges < 0 || n_edges > GNN_CSR_NOALLOC_MAX_EDGES || !rowptr)
    return GNN_ERR_INVALID_ARG;
  if (n_edges > 0 && (!edge_index || !perm || !src_sorted)) return GNN_ERR_INVALID_ARG;
  void* sp = nullptr;                             // device address of the scratch array (current context)
  cudaError_t ce = cudaGetSymbolAddress(&sp, g_csr_noalloc_scratch);
  if (ce != cudaSuccess) return cuda_fail(ce);
  unsigned char* scratch = static_cast<unsigned char*>(sp);
  cudaStream_t st = (cudaStream_t)stream;
  const int N = (int)n_nodes, E = (int)n_edges;
  const int tb = 256;
  if (E == 0) {                                   // every row pointer is 0
    csr_rowptr_kernel<<<blocks_for((int64_t)N + 1, tb), tb, 0, st>>>(nullptr, 0, N, rowptr);
    ce = cudaGetLastError();
    return ce == cudaSuccess ? GNN_OK : cuda_fail(ce);
  }
  int* words = reinterpret_cast<int*>(scratch);
  int* keys_a = words;
  int* keys_b = keys_a + GNN_CSR_NOALLOC_MAX_EDGES;
  int* vals_a = keys_b + GNN_CSR_NOALLOC_MAX_EDGES;
  int* vals_b = vals_a + GNN_CSR_NOALLOC_MAX_EDGES;
  int* src_c = vals_b + GNN_CSR_NOALLOC_MAX_EDGES;
  int* hist = src_c + GNN_CSR_NOALLOC_MAX_EDGES;
  csr_keys_kernel<<<blocks_for(E, tb), tb, 0, st>>>(edge_index, E, N, keys_a, vals_a, src_c, nullptr);
  int bits = 0;
  while (bits < 31 && (N >> bits) != 0) ++bits;   // keys lie in [0, N]
  if (bits == 0) bits = 1;
  const int passes = (bits + 7) / 8;
  const int tiles = (int)blocks_for(E, kRadixTile);
  int *kin = keys_a, *vin = vals_a, *kout = keys_b, *vout = vals_b;
  for (int ps = 0; ps < passes; ++ps) {
    const int shift = 8 * ps;
    radix_count_kernel<<<tiles, kRadixThreads, 0, st>>>(kin, E, shift, tiles, hist);
    radix_offsets_kernel<<<1, kOffsetsThreads, 0, st>>>(hist, tiles);
    radix_scatter_kernel<<<tiles, kRadixThreads, 0, st>>>(kin, vin, kout, vout, E, shift, tiles, hist);
    int* t = kin; kin = kout; kout = t;
    t = vin; vin = vout; vout = t;
  }
  // sorted keys in kin; kout is free and receives the (unused) clamped destinations
  csr_gather_kernel<<<blocks_for(E, tb), tb, 0, st>>>(kin, vin, src_c, E, N, perm, src_sorted, kout);
  csr_rowptr_kernel<<<blocks_for((int64_t)N + 1, tb), tb, 0, st>>>(kin, E, N, rowptr);
  ce = cudaGetLastError();
  return ce == cudaSuccess ? GNN_OK : cuda_fail(ce);
}
