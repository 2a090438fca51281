// Edge filtering's compaction step: keep the edges whose score is above a
// threshold, in input order (a stable, deterministic stream compaction).
//
// Blocks of 1024 edges: count the kept edges of every block, scan the block
// counts (one block), then each block writes its kept edges at its offset,
// ranked in input order (warp ballots within a round of 256 edges, warp totals
// across a round, a running count across rounds).  The output is the kept edge
// list [2, n_kept], contiguous (row 1 starts at n_kept), plus the input id of
// every kept edge.
#pragma once
#include <cstdint>

namespace gnn {

constexpr int kCompactThreads = 256;
constexpr int kCompactRounds = 4;
constexpr int kCompactBlock = kCompactThreads * kCompactRounds;   // edges per block

__device__ __forceinline__ bool kept(float score, float threshold) { return score > threshold; }  // NaN: no

__global__ void __launch_bounds__(kCompactThreads) compact_count_kernel(const float* __restrict__ scores, int m,
                                                                        float threshold, int* __restrict__ counts) {
  __shared__ int wsum[kCompactThreads / 32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  int c = 0;
#pragma unroll
  for (int r = 0; r < kCompactRounds; ++r) {
    const int k = blockIdx.x * kCompactBlock + r * kCompactThreads + t;
    c += (k < m && kept(scores[k], threshold)) ? 1 : 0;
  }
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 0) wsum[warp] = c;
  __syncthreads();
  if (t == 0) {
    int s = 0;
    for (int w = 0; w < kCompactThreads / 32; ++w) s += wsum[w];
    counts[blockIdx.x] = s;
  }
}

// Exclusive scan of the block counts in place (one block of 1024 threads); the total goes to *total.
// The sums are taken in 64 bits and the total saturates at INT32_MAX, so a caller that compares the
// total with its capacity (below INT32_MAX) sees an overflow as "too many" (offsets past the
// overflow point are then meaningless and must not be used).
__global__ void __launch_bounds__(1024) compact_scan_kernel(int* __restrict__ counts, int n_blocks,
                                                            int* __restrict__ total) {
  __shared__ long long wsum[32];
  __shared__ long long carry;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  if (t == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < n_blocks; base += 1024) {
    const int i = base + t;
    const long long v = i < n_blocks ? counts[i] : 0;
    long long x = v;                                       // inclusive scan inside the warp
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      long long w = wsum[lane];
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;                                      // inclusive over warps
    }
    __syncthreads();
    const long long excl = carry + (warp > 0 ? wsum[warp - 1] : 0) + x - v;
    if (i < n_blocks) counts[i] = (int)excl;
    __syncthreads();
    if (t == 0) carry += wsum[31];
    __syncthreads();
  }
  if (t == 0) *total = carry > 0x7fffffffLL ? 0x7fffffff : (int)carry;
}

// Exclusive scan of a long int array in place, in three launches: scan_reduce_kernel (sum of
// every 1024 entries, saturated at INT32_MAX), compact_scan_kernel over those sums (offsets and
// the total), scan_apply_kernel (offset plus the scan inside each 1024 entries).  A total above
// INT32_MAX saturates there; the offsets are then meaningless and the caller must not use them.
constexpr int kScanBlock = 1024;

__global__ void __launch_bounds__(kScanBlock) scan_reduce_kernel(const int* __restrict__ v, int n,
                                                                 int* __restrict__ sums) {
  __shared__ long long wsum[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int i = blockIdx.x * kScanBlock + t;
  long long x = i < n ? v[i] : 0;
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  if (lane == 0) wsum[warp] = x;
  __syncthreads();
  if (t == 0) {
    long long s = 0;
    for (int w = 0; w < 32; ++w) s += wsum[w];
    sums[blockIdx.x] = s > 0x7fffffffLL ? 0x7fffffff : (int)s;
  }
}

__global__ void __launch_bounds__(kScanBlock) scan_apply_kernel(int* __restrict__ v, int n,
                                                                const int* __restrict__ offsets) {
  __shared__ int wsum[32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int i = blockIdx.x * kScanBlock + t;
  const int c = i < n ? v[i] : 0;
  int x = c;
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = wsum[lane];
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    wsum[lane] = w;
  }
  __syncthreads();
  if (i < n) v[i] = offsets[blockIdx.x] + (warp > 0 ? wsum[warp - 1] : 0) + x - c;
}

__global__ void __launch_bounds__(kCompactThreads) compact_scatter_kernel(
    const float* __restrict__ scores, const int32_t* __restrict__ ei, int m, float threshold,
    const int* __restrict__ offsets, const int* __restrict__ total, int32_t* __restrict__ out_ei,
    int32_t* __restrict__ out_id) {
  __shared__ int wcnt[kCompactThreads / 32];
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int n_kept = *total;
  int run = offsets[blockIdx.x];
  for (int r = 0; r < kCompactRounds; ++r) {
    const int k = blockIdx.x * kCompactBlock + r * kCompactThreads + t;
    const bool keep = k < m && kept(scores[k], threshold);
    const unsigned ball = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) wcnt[warp] = __popc(ball);
    __syncthreads();
    int before = 0, round_total = 0;
#pragma unroll
    for (int w = 0; w < kCompactThreads / 32; ++w) {
      before += w < warp ? wcnt[w] : 0;
      round_total += wcnt[w];
    }
    if (keep) {
      const int pos = run + before + __popc(ball & ((1u << lane) - 1u));
      out_ei[pos] = ei[k];
      out_ei[(size_t)n_kept + pos] = ei[(size_t)m + k];
      if (out_id) out_id[pos] = k;
    }
    run += round_total;
    __syncthreads();
  }
}

}  // namespace gnn
