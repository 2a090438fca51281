// Track candidates from scored edges: weakly connected components of the edges
// whose score passes a threshold, labelled by the smallest hit id in each
// component (one integer label per space point).
//
// Lock-free union-find on the label array itself (no scratch): every link
// hangs the larger root under the smaller one, so parent[v] <= v always holds
// and each component's final root is its smallest member.  That makes the
// labels canonical: independent of thread order and of the order of the
// edges.  During the unions, path halving writes are plain stores; they race
// benignly because every value written is an ancestor of the node.  The final
// pass only reads the forest (see cc_flatten_kernel).
#pragma once
#include <cstdint>
#include "ptx.cuh"

namespace gnn {

// Wall-clock limit of the union and find loops (checked every 256 steps on %globaltimer, like
// every wait in the library); a loop that reaches it records DEV_ERR_TIMEOUT and gives up.
constexpr uint64_t kUnionLimitNs = 1000000000ull;   // 1 s

__global__ void cc_init_kernel(int32_t* parent, int n) {
  const int v = blockIdx.x * blockDim.x + threadIdx.x;
  if (v < n) parent[v] = v;
}

// Root of x, halving the path on the way.  Every parent is <= its child, so a walk ends after at
// most x steps; the time limit bounds it regardless.  Returns -1 when the limit expired.
__device__ __forceinline__ int cc_find(int32_t* parent, int x, uint64_t t0) {
  volatile int32_t* p = parent;
  for (uint32_t it = 1;; ++it) {
    const int px = p[x];
    if (px == x) return x;
    const int gx = p[px];
    if (gx != px) p[x] = gx;                           // path halving
    x = px;
    if ((it & 255u) == 0 && global_timer_ns() - t0 > kUnionLimitNs) return -1;
  }
}

// One thread per edge: unite the endpoints of every edge kept by the threshold.  Edges with an
// endpoint outside [0, n) and edges whose score is NaN or <= threshold are skipped.
__global__ void cc_union_kernel(const float* __restrict__ scores, const int32_t* __restrict__ ei, int n, int m,
                                float threshold, int32_t* parent, uint32_t* err) {
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= m) return;
  const float s = scores[k];
  if (!(s > threshold)) return;
  int u = ei[k], v = ei[(size_t)m + k];
  if (u < 0 || u >= n || v < 0 || v >= n) return;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 1;; ++it) {
    u = cc_find(parent, u, t0);
    v = u < 0 ? -1 : cc_find(parent, v, t0);
    if (v < 0 || ((it & 255u) == 0 && global_timer_ns() - t0 > kUnionLimitNs)) {
      atomicOr(err, DEV_ERR_TIMEOUT);
      return;
    }
    if (u == v) return;
    if (u < v) { const int t = u; u = v; v = t; }     // u: the larger root, hung under v
    if (atomicCAS(parent + u, u, v) == u) return;
  }
}

// Shortens the forest before the final pass: every node points at the root its (path-halving)
// walk reached.  Racing halving stores can leave some nodes one or more steps below their root,
// so this pass alone does not give the labels; it only makes the read-only walks short.
__global__ void cc_compress_kernel(int32_t* parent, int n, uint32_t* err) {
  const int v = blockIdx.x * blockDim.x + threadIdx.x;
  if (v >= n) return;
  const int r = cc_find(parent, v, global_timer_ns());
  if (r >= 0) parent[v] = r;
  else atomicOr(err, DEV_ERR_TIMEOUT);
}

// labels[v] = root of v (the smallest id of its component).  The walk only reads: a path-halving
// store from another thread could otherwise land on parent[v] after v has written its root and
// leave v pointing at an intermediate ancestor.  Every value a reader meets is an ancestor (an
// old parent or a final root), so each walk still ends at its root.
__global__ void cc_flatten_kernel(int32_t* parent, int n, uint32_t* err) {
  const int v = blockIdx.x * blockDim.x + threadIdx.x;
  if (v >= n) return;
  volatile int32_t* p = parent;
  const uint64_t t0 = global_timer_ns();
  int x = v;
  for (uint32_t it = 1;; ++it) {
    const int px = p[x];
    if (px == x) break;
    x = px;
    if ((it & 255u) == 0 && global_timer_ns() - t0 > kUnionLimitNs) {
      atomicOr(err, DEV_ERR_TIMEOUT);
      break;
    }
  }
  parent[v] = x;
}

}  // namespace gnn
