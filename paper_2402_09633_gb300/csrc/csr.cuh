// Destination-keyed CSR of the candidate edges, built on the device.
//
// The message-passing step sums every edge's message into its destination
// node.  Sorting the edges by destination turns that sum into a contiguous
// segment per node, read in a fixed order (deterministic, no float atomics),
// and lets the edge kernels stream the per-edge state in that order.
//
// Steps: validate endpoints and form keys (key = dst, or n_nodes for an edge
// with an endpoint out of range), stable LSD radix sort of (key, input id)
// with 8-bit digits, then gather the sources in sorted order and mark the
// first slot of every node (rowptr).  A stable sort of keys that only differ
// in input id gives the unique order "by destination, then input id".
#pragma once
#include <cstdint>
#include "ptx.cuh"

namespace gnn {

constexpr int kRadixThreads = 256;
constexpr int kRadixRounds = 16;
constexpr int kRadixTile = kRadixThreads * kRadixRounds;   // elements per tile

// K0: endpoint validation and sort keys.  An out-of-range edge sets DEV_ERR_INDEX_RANGE in *err
// (when err is not null) and sorts last (key n_nodes).
__global__ void csr_keys_kernel(const int32_t* __restrict__ ei, int n_edges, int n_nodes,
                                int* __restrict__ keys, int* __restrict__ vals,
                                int* __restrict__ src_clamped, uint32_t* err) {
  pdl_wait();
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= n_edges) return;
  const int s = ei[k];
  const int d = ei[(size_t)n_edges + k];
  const bool ok = (s >= 0) & (s < n_nodes) & (d >= 0) & (d < n_nodes);
  keys[k] = ok ? d : n_nodes;
  vals[k] = k;
  src_clamped[k] = ok ? s : 0;
  if (!ok && err) atomicOr(err, DEV_ERR_INDEX_RANGE);
}

// Per-tile digit histogram: hist[tile * 256 + digit].
__global__ void radix_count_kernel(const int* __restrict__ keys, int n, int shift, int n_tiles,
                                   int* __restrict__ hist) {
  pdl_wait();
  __shared__ int cnt[256];
  cnt[threadIdx.x] = 0;
  __syncthreads();
  const int base = blockIdx.x * kRadixTile;
  for (int i = threadIdx.x; i < kRadixTile; i += kRadixThreads) {
    const int idx = base + i;
    if (idx < n) atomicAdd(&cnt[(keys[idx] >> shift) & 255], 1);
  }
  __syncthreads();
  hist[blockIdx.x * 256 + threadIdx.x] = cnt[threadIdx.x];
}

// Scatter offsets of one radix pass, in place: hist[tile * 256 + d] becomes the
// number of keys with a smaller digit (all tiles) plus those with digit d in
// earlier tiles.  One block of kOffsetsThreads: thread (part, d) owns digit d
// over one contiguous quarter of the tiles (reads coalesced across digits) and
// keeps kOffsetsBatch loads in flight; the quarters' sums and the 256 digit
// totals are combined in shared memory.  (A single thread per digit walking
// every tile with one dependent load at a time took 23 us per pass.)
constexpr int kOffsetsThreads = 1024;
constexpr int kOffsetsParts = kOffsetsThreads / 256;
constexpr int kOffsetsBatch = 16;
__global__ void __launch_bounds__(kOffsetsThreads) radix_offsets_kernel(int* __restrict__ hist, int n_tiles) {
  pdl_wait();
  __shared__ int part_sum[kOffsetsParts][256];
  __shared__ int tot[256];
  const int d = threadIdx.x & 255, part = threadIdx.x >> 8;
  const int per = (n_tiles + kOffsetsParts - 1) / kOffsetsParts;
  const int t0 = part * per, t1 = min(n_tiles, t0 + per);
  int sum = 0;
  for (int t = t0; t < t1; t += kOffsetsBatch) {            // pass 1: this quarter's count of digit d
    int v[kOffsetsBatch];
#pragma unroll
    for (int i = 0; i < kOffsetsBatch; ++i) v[i] = t + i < t1 ? hist[(t + i) * 256 + d] : 0;
#pragma unroll
    for (int i = 0; i < kOffsetsBatch; ++i) sum += v[i];
  }
  part_sum[part][d] = sum;
  __syncthreads();
  if (part == 0) {
    int all = 0;
#pragma unroll
    for (int k = 0; k < kOffsetsParts; ++k) all += part_sum[k][d];
    tot[d] = all;
  }
  __syncthreads();
  for (int off = 1; off < 256; off <<= 1) {                  // inclusive scan of the digit totals
    const int v = (part == 0 && d >= off) ? tot[d - off] : 0;
    __syncthreads();
    if (part == 0) tot[d] += v;
    __syncthreads();
  }
  int run = d > 0 ? tot[d - 1] : 0;                          // keys with a smaller digit
  for (int k = 0; k < part; ++k) run += part_sum[k][d];      // digit d in earlier quarters
  for (int t = t0; t < t1; t += kOffsetsBatch) {            // pass 2: exclusive offsets
    int v[kOffsetsBatch];
#pragma unroll
    for (int i = 0; i < kOffsetsBatch; ++i) v[i] = t + i < t1 ? hist[(t + i) * 256 + d] : 0;
#pragma unroll
    for (int i = 0; i < kOffsetsBatch; ++i)
      if (t + i < t1) { hist[(t + i) * 256 + d] = run; run += v[i]; }
  }
}

// Stable scatter of one radix pass.  Elements of a tile are ranked in input
// order: round r handles elements [r*256, r*256+256); within a warp the rank
// among equal digits comes from __match_any_sync, across warps from per-warp
// digit counts, across rounds from a running per-digit counter.
__global__ void radix_scatter_kernel(const int* __restrict__ keys_in, const int* __restrict__ vals_in,
                                     int* __restrict__ keys_out, int* __restrict__ vals_out, int n,
                                     int shift, int n_tiles, const int* __restrict__ offs) {
  pdl_wait();
  __shared__ int run[256];
  __shared__ int wcnt[kRadixThreads / 32][256];
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  run[t] = offs[blockIdx.x * 256 + t];
  const int base = blockIdx.x * kRadixTile;
  const unsigned lt_mask = (1u << lane) - 1u;
  for (int r = 0; r < kRadixRounds; ++r) {
    const int idx = base + r * kRadixThreads + t;
    const bool has = idx < n;
    const int key = has ? keys_in[idx] : 0;
    const int val = has ? vals_in[idx] : 0;
    const int dig = has ? ((key >> shift) & 255) : 256;
#pragma unroll
    for (int w = 0; w < kRadixThreads / 32; ++w) wcnt[w][t] = 0;
    __syncthreads();
    const unsigned peers = __match_any_sync(0xffffffffu, dig);
    const int rank = __popc(peers & lt_mask);
    if (has && rank == 0) wcnt[warp][dig] = __popc(peers);
    __syncthreads();
    if (has) {
      int pos = run[dig] + rank;
      for (int w = 0; w < warp; ++w) pos += wcnt[w][dig];
      keys_out[pos] = key;
      vals_out[pos] = val;
    }
    __syncthreads();
    int add = 0;
#pragma unroll
    for (int w = 0; w < kRadixThreads / 32; ++w) add += wcnt[w][t];
    run[t] += add;
    __syncthreads();
  }
}

// Sorted order -> perm, src_sorted, dst_sorted (clamped for invalid edges).
__global__ void csr_gather_kernel(const int* __restrict__ keys_sorted, const int* __restrict__ vals_sorted,
                                  const int* __restrict__ src_clamped, int n_edges, int n_nodes,
                                  int* __restrict__ perm, int* __restrict__ src_sorted,
                                  int* __restrict__ dst_sorted) {
  pdl_wait();
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= n_edges) return;
  const int id = vals_sorted[k];
  const int key = keys_sorted[k];
  perm[k] = id;
  src_sorted[k] = src_clamped[id];
  dst_sorted[k] = key < n_nodes ? key : 0;
}

// rowptr[j] = first sorted slot whose key >= j (binary search), for j in [0, n_nodes].
__global__ void csr_rowptr_kernel(const int* __restrict__ keys_sorted, int n_edges, int n_nodes,
                                  int* __restrict__ rowptr) {
  pdl_wait();
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j > n_nodes) return;
  int lo = 0, hi = n_edges;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (keys_sorted[mid] < j) lo = mid + 1; else hi = mid;
  }
  rowptr[j] = lo;
}

}  // namespace gnn
