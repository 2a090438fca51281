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
// The counting pass also keeps the partners it finds, in the order it finds
// them, in a chain of 64-byte chunks per hit (its own first chunk, further ones
// from a pool), so the writing pass copies instead of searching again; a hit
// whose chain could not grow (pool exhausted) is searched again.
#pragma once
#include <climits>
#include <cstdint>
#include "ptx.cuh"

namespace gnn {

constexpr int kFrnnReach = 2;            // cells a partner can lie away on each axis
constexpr int kFrnnChunk = 16;           // ints per partner chunk: 15 sorted positions + the next chunk
constexpr int kFrnnLost = -2;            // link of a hit's first chunk: chain incomplete, search again

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

// The candidate loop over one run of sorted positions [p, p1).  Candidates are tested 32 at a time into a bit mask (the distance loop stays free of the rare
// work of a hit, so nothing of it is executed predicated for every candidate); the partners found
// are then taken in ascending position: written (writing pass) or counted and kept in the chain.
// Measured on the full event: appending inside the distance loop made the counting pass ~60 %
// slower.
#define GNN_FRNN_RUN()                                                                                   \
  for (; p < p1; p += 32) {                                                                              \
    const int pe = p1 - p < 32 ? p1 : p + 32;                                                            \
    uint32_t hits = 0;                                                                                   \
    for (int pp = p; pp < pe; ++pp) {                                                                    \
      float s = 0.f;                                                                                     \
      _Pragma("unroll") for (int c = 0; c < CH; ++c) {                                                   \
        const float4 e = emb_s[(size_t)pp * CH + c];                                                     \
        s = frnn_acc(s, q[c].x, e.x);                                                                    \
        s = frnn_acc(s, q[c].y, e.y);                                                                    \
        s = frnn_acc(s, q[c].z, e.z);                                                                    \
        s = frnn_acc(s, q[c].w, e.w);                                                                    \
      }                                                                                                  \
      hits |= (s < r2 ? 1u : 0u) << (pp - p);                                                            \
    }                                                                                                    \
    while (hits) {                                                                                       \
      const int pf = p + __ffs(hits) - 1;                                                                \
      hits &= hits - 1;                                                                                  \
      if (write) {                                                                                       \
        emit(pf);                                                                                        \
      } else {                                                                                           \
        ++found;                                                                                         \
        if (!lost) {                                                                                     \
          if (fill == kFrnnChunk - 1) {                                                                  \
            const int nc = atomicAdd(next_chunk, 1);                                                     \
            if (nc >= max_extra) {                                                                       \
              lost = true;                                                                               \
            } else {                                                                                     \
              chunks[(size_t)cur * kFrnnChunk + kFrnnChunk - 1] = n + nc;                                \
              cur = n + nc;                                                                              \
              fill = 0;                                                                                  \
            }                                                                                            \
          }                                                                                              \
          if (!lost) chunks[(size_t)cur * kFrnnChunk + fill++] = pf;                                     \
        }                                                                                                \
      }                                                                                                  \
    }                                                                                                    \
  }

// One thread per sorted position t.  write == 0: counts[t] = pairs visited from t, the partners kept
// in t's chain; write == 1: the pairs of the hits whose chain was lost, at offsets[t] (exclusive scan
// of counts), when the total fits (frnn_copy_kernel writes the others).  (Measured on the full event,
// before the chains: separate counting and writing kernels, or a block-level scan of the counts
// inside this kernel, made the search 12-22 % slower; the scan runs as separate kernels between the
// passes instead.)
constexpr int kFrnnPairsThreads = 128;   // 3 % faster than 256 on the full event (shorter tail)

// The pairs of every hit whose chain was kept: the partners' sorted positions, read a chunk at a
// time, with their hit ids and r gathered together, written oriented from the smaller r.
__global__ void __launch_bounds__(256) frnn_copy_kernel(const float* __restrict__ r_s, int n,
                                                        const int* __restrict__ ids, const int* __restrict__ offsets,
                                                        const int* __restrict__ total, int capacity,
                                                        const int* __restrict__ chunks, int32_t* __restrict__ out) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  const int n_total = *total;
  if (n_total > capacity || chunks[(size_t)t * kFrnnChunk + kFrnnChunk - 1] == kFrnnLost) return;
  int pos = offsets[t];
  const int cnt = (t + 1 < n ? offsets[t + 1] : n_total) - pos;
  const int i = ids[t];
  const float ri = r_s[t];
  int cur = t;
  for (int base = 0; base < cnt; base += kFrnnChunk - 1) {
    const int4* c4 = reinterpret_cast<const int4*>(chunks + (size_t)cur * kFrnnChunk);
    const int4 w0 = c4[0], w1 = c4[1], w2 = c4[2], w3 = c4[3];
    const int w[kFrnnChunk] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w,
                               w2.x, w2.y, w2.z, w2.w, w3.x, w3.y, w3.z, w3.w};
    const int m = cnt - base;
    int jj[kFrnnChunk - 1];
    float rr[kFrnnChunk - 1];
#pragma unroll
    for (int k = 0; k < kFrnnChunk - 1; ++k) {
      jj[k] = k < m ? ids[w[k]] : 0;
      rr[k] = k < m ? r_s[w[k]] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < kFrnnChunk - 1; ++k) {
      if (k < m) {
        const bool i_first = ri < rr[k] || (ri == rr[k] && i < jj[k]);
        out[pos] = i_first ? i : jj[k];
        out[(size_t)n_total + pos] = i_first ? jj[k] : i;
        ++pos;
      }
    }
    cur = w[kFrnnChunk - 1];
  }
}

// chunks: [n + max_extra][kFrnnChunk] ints; chunk t is hit t's first, pool chunks follow (next_chunk
// counts those taken, from zero).
template <int CH, int K>
__global__ void __launch_bounds__(kFrnnPairsThreads) frnn_pairs_kernel(
    const float4* __restrict__ emb_s, const float* __restrict__ r_s, int n, float r2, int grid,
    const int* __restrict__ cell_keys, const int* __restrict__ ids, const int* __restrict__ cell_start, int write,
    int* __restrict__ counts, const int* __restrict__ total, int capacity, int32_t* __restrict__ out,
    int* __restrict__ chunks, int* __restrict__ next_chunk, int max_extra, uint32_t* err) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= n) return;
  int pos = 0, n_total = 0;
  int i = 0;
  float ri = 0.f;
  auto emit = [&](int p) {
    const int j = ids[p];
    const float rj = r_s[p];
    const bool i_first = ri < rj || (ri == rj && i < j);
    out[pos] = i_first ? i : j;
    out[(size_t)n_total + pos] = i_first ? j : i;
    ++pos;
  };
  if (write) {
    n_total = *total;
    if (n_total > capacity) {
      if (t == 0) atomicOr(err, DEV_ERR_CAPACITY);
      return;
    }
    pos = counts[t];
    i = ids[t];
    ri = r_s[t];
    if (chunks[(size_t)t * kFrnnChunk + kFrnnChunk - 1] != kFrnnLost) return;   // frnn_copy_kernel's
  }
  int cur = t, fill = 0;                         // counting pass: the chain being filled
  bool lost = false;
  if (!write) chunks[(size_t)t * kFrnnChunk + kFrnnChunk - 1] = -1;   // link of the first chunk: none yet
  float4 q[CH];
#pragma unroll
  for (int c = 0; c < CH; ++c) q[c] = emb_s[(size_t)t * CH + c];
  int key = cell_keys[t];
  const int cl = key % grid;                     // last gridded coordinate: the run axis
  key /= grid;
  const int lo = cl - kFrnnReach < 0 ? 0 : cl - kFrnnReach;
  const int hi = cl + kFrnnReach >= grid ? grid - 1 : cl + kFrnnReach;
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
  if (!write) {
    counts[t] = found;
    if (lost) chunks[(size_t)t * kFrnnChunk + kFrnnChunk - 1] = kFrnnLost;
  }
}
#undef GNN_FRNN_RUN

}  // namespace gnn
