// Graph construction in the embedding space: every pair of hits whose
// embeddings lie within a fixed radius becomes a candidate edge (fixed-radius
// nearest neighbours).
//
// The embeddings are unit vectors, so each coordinate lies in [-1, 1].  Hits
// are binned on a uniform grid over their first three coordinates with cells
// wider than the radius (a coordinate outside [-1, 1] is clamped to the edge
// cells, which keeps the search exact, only slower), and sorted by cell (the library's stable radix
// sort).  Each hit then visits the 27 cells around its own and tests the full
// D-dimensional squared distance, summed over the coordinates in order with one
// rounding per product and per sum (no fused multiply-add), against radius^2
// rounded to fp32.  A pair is found once, by its hit with the smaller index,
// and oriented from the hit with the smaller r (column 0 of the node features,
// index as tie-break) to the other.  A counting pass, a scan and a writing pass
// make the output order deterministic: by the finding hit's position in the
// cell order, then by cell and position of the partner.
#pragma once
#include <cstdint>
#include "ptx.cuh"

namespace gnn {

constexpr int kFrnnMaxGrid = 128;        // cells per axis

// Cells per axis: cells a little wider than the radius (0.1 % margin), so that the rounding of the
// cell coordinates and of the distance test never puts a pair within the radius two cells apart.
__host__ __device__ inline int frnn_grid(float radius) {
  const float cells = 1.998f / radius;
  return cells >= (float)kFrnnMaxGrid ? kFrnnMaxGrid : (cells < 1.0f ? 1 : (int)cells);
}

__device__ __forceinline__ int frnn_coord(float e, int grid) {
  int c = (int)floorf((e + 1.0f) * 0.5f * (float)grid);
  return c < 0 ? 0 : (c >= grid ? grid - 1 : c);
}

__global__ void frnn_cell_kernel(const float* __restrict__ emb, int n, int dim, int grid, int* __restrict__ keys,
                                 int* __restrict__ vals) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float* e = emb + (size_t)i * dim;
  const int c0 = frnn_coord(e[0], grid);
  const int c1 = dim > 1 ? frnn_coord(e[1], grid) : 0;
  const int c2 = dim > 2 ? frnn_coord(e[2], grid) : 0;
  keys[i] = (c0 * grid + c1) * grid + c2;
  vals[i] = i;
}

// One thread per sorted position t (hit i = ids[t]).  write == 0: counts[t] = pairs found by i;
// write == 1: those pairs at offsets[t] (exclusive scan of counts), when the total fits.
__global__ void frnn_pairs_kernel(const float* __restrict__ emb, const float* __restrict__ x, int x_stride, int n,
                                  int dim, float r2, int grid, const int* __restrict__ cell_keys,
                                  const int* __restrict__ ids, const int* __restrict__ cell_start, int write,
                                  int* __restrict__ counts, const int* __restrict__ total, int capacity,
                                  int32_t* __restrict__ out, uint32_t* err) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const int i = ids[t];
  float ei[16];
#pragma unroll
  for (int d = 0; d < 16; ++d) ei[d] = d < dim ? emb[(size_t)i * dim + d] : 0.f;
  const int key = cell_keys[t];
  const int c2 = key % grid, c1 = (key / grid) % grid, c0 = key / (grid * grid);
  int found = 0, pos = 0, n_total = 0;
  if (write) {
    n_total = *total;
    if (n_total > capacity) {
      if (t == 0) atomicOr(err, DEV_ERR_CAPACITY);
      return;
    }
    pos = counts[t];
  }
  const float ri = write ? x[(size_t)i * x_stride] : 0.f;
  for (int a = c0 - 1; a <= c0 + 1; ++a) {
    if (a < 0 || a >= grid) continue;
    for (int b = c1 - 1; b <= c1 + 1; ++b) {
      if (b < 0 || b >= grid) continue;
      for (int c = c2 - 1; c <= c2 + 1; ++c) {
        if (c < 0 || c >= grid) continue;
        const int cell = (a * grid + b) * grid + c;
        for (int q = cell_start[cell], q1 = cell_start[cell + 1]; q < q1; ++q) {
          const int j = ids[q];
          if (j <= i) continue;
          const float* ej = emb + (size_t)j * dim;
          float s = 0.f;                       // no fused multiply-add: one rounding per product and sum
#pragma unroll
          for (int d = 0; d < 16; ++d) {
            if (d < dim) {
              const float diff = ei[d] - ej[d];
              s = __fadd_rn(s, __fmul_rn(diff, diff));
            }
          }
          if (!(s < r2)) continue;
          if (write) {
            const float rj = x[(size_t)j * x_stride];
            const bool i_first = ri < rj || (ri == rj && i < j);
            out[pos] = i_first ? i : j;
            out[(size_t)n_total + pos] = i_first ? j : i;
            ++pos;
          } else {
            ++found;
          }
        }
      }
    }
  }
  if (!write) counts[t] = found;
}

}  // namespace gnn
