// Graph construction in the embedding space: every pair of hits whose
// embeddings lie within a fixed radius becomes a candidate edge (fixed-radius
// nearest neighbours).
//
// The embeddings are unit vectors, so each coordinate lies in [-1, 1].  Hits
// are binned on a uniform grid over their first K coordinates (K = 4 when the
// embedding has at least 4, else 3) with cells a little wider than half the
// radius (a coordinate outside [-1, 1] is clamped to the edge cells, which
// keeps the search exact, only slower), and sorted by cell (the library's
// stable radix sort); their embeddings and r values are then gathered into
// that order, zero-padded to a multiple of four coordinates.  A pair within
// the radius lies at most two cells apart on each axis, so the partners of a
// hit sit in the 5^(K-1) "rows" of cells around its own (rows over the first
// K-1 gridded coordinates), and in each row in one run of at most five
// consecutive cells along the last one, which is one contiguous range of
// sorted positions.  Rows before the hit's own row hold only earlier positions:
// each pair is visited once, by its earlier sorted position, which scans
// (5^(K-1) + 1) / 2 rows (its own row from the next position on).
//
// The test is the full squared distance, summed over the coordinates in order
// with one rounding per product and per sum (no fused multiply-add; the zero
// padding adds exact zeros), against radius^2 rounded to fp32.  Each pair
// becomes one edge, oriented from the hit with the smaller r (column 0 of the
// node features, hit id as tie-break).  A counting pass, an exclusive scan of
// the per-hit counts and a writing pass make the output order deterministic: by
// the visiting hit's sorted position, then by row and position of the partner.
#pragma once
#include <cstdint>
#include "ptx.cuh"

namespace gnn {

constexpr int kFrnnReach = 2;            // cells a partner can lie away on each axis

// Cells per axis for a grid over K coordinates (K = 3 or 4): cells 0.1 % wider than half the radius,
// so that the rounding of the cell coordinates and of the distance test never puts a pair within
// the radius three cells apart; at most 128 (K = 3) or 64 (K = 4) cells per axis.
__host__ __device__ inline int frnn_grid(float radius, int K) {
  const int max_grid = K == 4 ? 64 : 128;
  const float cells = 1.998f * (float)kFrnnReach / radius;
  return cells >= (float)max_grid ? max_grid : (cells < 1.0f ? 1 : (int)cells);
}

__device__ __forceinline__ int frnn_coord(float e, int grid) {
  int c = (int)floorf((e + 1.0f) * 0.5f * (float)grid);
  return c < 0 ? 0 : (c >= grid ? grid - 1 : c);
}

// Cell key of every hit: its cell over the first K coordinates (missing ones count as cell 0),
// row-major with the last gridded coordinate fastest.
template <int K>
__global__ void frnn_cell_kernel(const float* __restrict__ emb, int n, int dim, int grid, int* __restrict__ keys,
                                 int* __restrict__ vals) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float* e = emb + (size_t)i * dim;
  int key = 0;
#pragma unroll
  for (int k = 0; k < K; ++k) key = key * grid + (k < dim ? frnn_coord(e[k], grid) : 0);
  keys[i] = key;
  vals[i] = i;
}

// Sorted copies: emb_s [n, 4 * CH] (zero-padded), r_s [n] = x[ids[t], 0].
template <int CH>
__global__ void frnn_gather_kernel(const float* __restrict__ emb, const float* __restrict__ x, int x_stride, int n,
                                   int dim, const int* __restrict__ ids, float4* __restrict__ emb_s,
                                   float* __restrict__ r_s) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const int i = ids[t];
  const float* e = emb + (size_t)i * dim;
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    float v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = 4 * c + k < dim ? e[4 * c + k] : 0.f;
    emb_s[(size_t)t * CH + c] = make_float4(v[0], v[1], v[2], v[3]);
  }
  r_s[t] = x[(size_t)i * x_stride];
}

__device__ __forceinline__ float frnn_acc(float s, float a, float b) {
  const float d = a - b;
  return __fadd_rn(s, __fmul_rn(d, d));
}

// One thread per sorted position t.  write == 0: counts[t] = pairs visited from t;
// write == 1: those pairs at offsets[t] (exclusive scan of counts), when the total fits.
// (Measured on the full event: separate counting and writing kernels, or a block-level scan of
// the counts inside this kernel, made the search 12-22 % slower; the scan runs as separate
// kernels between the passes instead.)
// The candidate loop over one run of sorted positions [p, p1).
#define GNN_FRNN_RUN()                                                                                   \
  for (; p < p1; ++p) {                                                                                  \
    float s = 0.f;                                                                                       \
    _Pragma("unroll") for (int c = 0; c < CH; ++c) {                                                     \
      const float4 e = emb_s[(size_t)p * CH + c];                                                        \
      s = frnn_acc(s, q[c].x, e.x);                                                                      \
      s = frnn_acc(s, q[c].y, e.y);                                                                      \
      s = frnn_acc(s, q[c].z, e.z);                                                                      \
      s = frnn_acc(s, q[c].w, e.w);                                                                      \
    }                                                                                                    \
    if (!(s < r2)) continue;                                                                             \
    if (write) {                                                                                         \
      const int j = ids[p];                                                                              \
      const float rj = r_s[p];                                                                           \
      const bool i_first = ri < rj || (ri == rj && i < j);                                               \
      out[pos] = i_first ? i : j;                                                                        \
      out[(size_t)n_total + pos] = i_first ? j : i;                                                      \
      ++pos;                                                                                             \
    } else {                                                                                             \
      ++found;                                                                                           \
    }                                                                                                    \
  }

// One thread per sorted position t.  write == 0: counts[t] = pairs visited from t;
// write == 1: those pairs at offsets[t] (exclusive scan of counts), when the total fits.
// (Measured on the full event: separate counting and writing kernels, or a block-level scan of
// the counts inside this kernel, made the search 12-22 % slower; the scan runs as separate
// kernels between the passes instead.)
constexpr int kFrnnPairsThreads = 128;   // 3 % faster than 256 on the full event (shorter tail)

template <int CH, int K>
__global__ void __launch_bounds__(kFrnnPairsThreads) frnn_pairs_kernel(
    const float4* __restrict__ emb_s, const float* __restrict__ r_s, int n, float r2, int grid,
    const int* __restrict__ cell_keys, const int* __restrict__ ids, const int* __restrict__ cell_start, int write,
    int* __restrict__ counts, const int* __restrict__ total, int capacity, int32_t* __restrict__ out,
    uint32_t* err) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  int pos = 0, n_total = 0;
  if (write) {
    n_total = *total;
    if (n_total > capacity) {
      if (t == 0) atomicOr(err, DEV_ERR_CAPACITY);
      return;
    }
    pos = counts[t];
  }
  float4 q[CH];
#pragma unroll
  for (int c = 0; c < CH; ++c) q[c] = emb_s[(size_t)t * CH + c];
  int key = cell_keys[t];
  const int cl = key % grid;                     // last gridded coordinate: the run axis
  key /= grid;
  const int lo = cl - kFrnnReach < 0 ? 0 : cl - kFrnnReach;
  const int hi = cl + kFrnnReach >= grid ? grid - 1 : cl + kFrnnReach;
  int i = 0;
  float ri = 0.f;
  if (write) { i = ids[t]; ri = r_s[t]; }
  int found = 0;
  if constexpr (K == 3) {
    const int c1 = key % grid, c0 = key / grid;
    for (int a = 0; a <= kFrnnReach; ++a) {
      const int ra = c0 + a;
      if (ra >= grid) break;
      for (int b = (a == 0 ? 0 : -kFrnnReach); b <= kFrnnReach; ++b) {
        const int rb = c1 + b;
        if (rb < 0 || rb >= grid) continue;
        const int row = (ra * grid + rb) * grid;
        int p = cell_start[row + lo];
        const int p1 = cell_start[row + hi + 1];
        if (a == 0 && b == 0) p = t + 1;
        GNN_FRNN_RUN()
      }
    }
  } else {
    const int c2 = key % grid, c1 = (key / grid) % grid, c0 = key / (grid * grid);
    for (int a = 0; a <= kFrnnReach; ++a) {
      const int ra = c0 + a;
      if (ra >= grid) break;
      for (int b = (a == 0 ? 0 : -kFrnnReach); b <= kFrnnReach; ++b) {
        const int rb = c1 + b;
        if (rb < 0 || rb >= grid) continue;
        for (int c = (a == 0 && b == 0 ? 0 : -kFrnnReach); c <= kFrnnReach; ++c) {
          const int rc = c2 + c;
          if (rc < 0 || rc >= grid) continue;
          const int row = ((ra * grid + rb) * grid + rc) * grid;
          int p = cell_start[row + lo];
          const int p1 = cell_start[row + hi + 1];
          if (a == 0 && b == 0 && c == 0) p = t + 1;
          GNN_FRNN_RUN()
        }
      }
    }
  }
  if (!write) counts[t] = found;
}
#undef GNN_FRNN_RUN

}  // namespace gnn
