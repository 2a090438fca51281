// Fused MLP-tile kernels of the interaction network (tcgen05 / TMEM, sm_103a).
//
// One persistent CTA per SM walks 128-row tiles (edges in destination-sorted
// CSR order, or nodes).  Each tile runs a fixed program of "jobs": a job is one
// Linear layer D = A * W^T executed on the 5th-generation tensor cores with
// the activation tile A in tensor memory and the weight W in shared memory,
// followed by an epilogue in registers (bias or gathered projections,
// LayerNorm, ReLU) that writes the next layer's A back into tensor memory.
//
// Precision (template parameter BF):
//   * fp32 model (BF = false): fp32 weights and states; every product is
//     evaluated as hi*hi + hi*lo + lo*hi of bf16 splits (v = hi + lo, both bf16)
//     with fp32 accumulation, which keeps the relative product error near 2^-16;
//   * bf16 model (BF = true): bf16 weights, bf16 activations and stored states
//     (e, h, a), one bf16 product per K step, fp32 accumulation and fp32
//     LayerNorm; the first-layer projections P_s, P_d stay fp32 (they are
//     partial sums of one Linear layer).
//
// Organisation (640 threads = 20 warps, one CTA per SM; setmaxnreg moves the
// control warpgroup's registers to the workers):
//   * two TMEM slots, each a D accumulator and a bf16 hi/lo A operand; slot s
//     works on tile 2p+s of tile pair p, so while one slot runs its epilogue
//     the tensor core serves the other (ping-pong);
//   * control warpgroup (warps 0-3): warp 0 issues the MMAs of whichever slot
//     has published its next A operand (one thread, 24 tcgen05.mma per layer)
//     and commits them to the slot's mbarrier; warp 1 loads the weights with
//     bulk copies (all at once, or streamed through a ring of stages);
//   * worker warpgroups (warps 4-19), eight warps per slot: a worker warp owns
//     16 rows of a tile; a quad of threads shares two rows (each thread a
//     quarter of the columns), reads them from tensor memory with the 16-lane
//     shapes and does bias / gathers, LayerNorm and ReLU in registers; one
//     worker thread per slot warms L2 (bulk prefetch) with the slot's next
//     tile a few microseconds before it is loaded.
#pragma once
#include <climits>
#include <cstdint>
#include <type_traits>
#include <cuda_bf16.h>
#include "ptx.cuh"

namespace gnn {

enum class TileKind : int {
  NodeEncoder = 0,     // x -> h0 (layer 1 on CUDA cores), then P_s, P_d projections
  EdgeEncoder = 1,     // (dr, dphi) -> e0 (layer 1 on CUDA cores)
  EdgeUpdate  = 2,     // e <- MLP_edge([h_src, h_dst, e]) via e*W_e + P_s[src] + P_d[dst]
  NodeUpdate  = 3,     // h <- MLP_node([h, sum of incoming e]); then P_s, P_d of new h
  Classifier  = 4,     // score = sigmoid(w_o . MLP_cls([h_src, h_dst, e]) + b_o)
  Filter      = 5,     // filtering step: score = sigmoid(w_o . MLP_f([x_src, x_dst]) + b_o), input edge order
  Embed       = 6,     // embedding step: y = normalize(W_out . MLP_emb(x) + b_out), D outputs per hit
};

constexpr int kMaxEmbedDim = 16;

constexpr int kThreads = 640;
// Register split (setmaxnreg): launch at 96 per thread (640 threads x 96 = 61440);
// the control warpgroup keeps 64 (the MMA issuer's and the weight producer's
// loop state must not spill: with ~200 KB of shared memory the L1 is small and
// a spilled value comes back from L2), the four worker warpgroups take 104:
// 128 x 64 + 512 x 104 = 61440.
constexpr int kControlRegs = 64;
constexpr int kWorkerRegs = 104;
static_assert(128 * kControlRegs + 512 * kWorkerRegs <= kThreads * 96, "register split exceeds the launch budget");
constexpr int kTileRows = 128;
constexpr int kMaxJobs = 8;

struct TileParams {
  int n_rows;                 // rows of this kernel: edges (E) or nodes (N)
  int n_tiles;
  int n_nodes;
  int n_layers;               // Linear layers per MLP (L)
  int n_feat;                 // encoder input width (F_n or 2)
  int n_jobs;
  int job_mat[kMaxJobs];      // matrix index (into wmats) of each MMA job
  int job_acc[kMaxJobs];      // 1: accumulate into D (second half of a split layer 1)
  const uint8_t* wmats;       // packed matrices, mat_bytes apart (hi part then lo part)
  uint32_t mat_bytes;
  const float* vecs;          // per-kernel fp32 parameter vectors (layout per kind)
  int n_vec_floats;
  float eps;
  // graph data
  const float* x;             // [N, n_feat_total] node features
  int x_stride;
  const int* src_sorted;      // [E] source of CSR slot k
  const int* dst_sorted;      // [E] destination of CSR slot k (clamped to a valid id)
  const int* key_sorted;      // [E] destination key (== n_nodes for an invalid edge)
  const int* perm;            // [E] input edge id of CSR slot k
  const int* rowptr;          // [N+1]
  void* e;                    // [E, H] edge state, CSR order (updated in place); fp32 or bf16
  void* h;                    // [N, H] node state; fp32 or bf16
  float* ps;                  // [N, H] projections W_s h
  float* pd;                  // [N, H] projections W_d h + b1
  void* agg;                  // [N, H] row-tiled: sum of incoming messages per node; fp32 or bf16
  float* scores;              // [E] input order
  uint32_t* err;              // device error word
  const int32_t* ei_in;       // filter: [2, E] input edge index (rows in input order)
  float* emb;                 // embedding: [N, emb_dim] output
  int emb_dim;
#ifdef GNN_TRACE
  unsigned long long* trace;  // [3 roles][kTraceEvents] %globaltimer stamps of CTA 0
#endif
};

#ifdef GNN_TRACE
constexpr int kTraceEvents = 512;
#define GNN_TRACE_AT(role, idx)                                                               \
  do {                                                                                        \
    if (p.trace && blockIdx.x == 0 && (idx) < kTraceEvents) p.trace[(role) * kTraceEvents + (idx)] = global_timer_ns(); \
  } while (0)
#define GNN_TRACE_W(label)                                                                   \
  do {                                                                                       \
    if (slot == 0 && trow == 0) GNN_TRACE_AT(1, tr_iter * 16 + (label));                     \
  } while (0)
#else
#define GNN_TRACE_AT(role, idx) do { } while (0)
#define GNN_TRACE_W(label) do { } while (0)
#endif

template <int H, bool BF>
struct TileGeom {
  static constexpr int HH = H / 2;                  // columns per worker thread
  static constexpr int SLOT_COLS = 2 * H;           // D (H cols) + A_hi (H/2) + A_lo (H/2, fp32 model only)
  static constexpr int TMEM_COLS = 2 * SLOT_COLS;   // two slots: 256 (H=64) or 512 (H=128)
  static constexpr uint32_t PART_BYTES = H * H * 2; // one bf16 H x H matrix part
  static constexpr uint32_t MAT_BYTES = BF ? PART_BYTES : 2 * PART_BYTES;  // hi [+ lo]
  static constexpr int STAGES = (192u * 1024u / MAT_BYTES) < 8 ? (192u * 1024u / MAT_BYTES) : 8;  // weight ring depth
  static constexpr uint32_t RING_BYTES = STAGES * MAT_BYTES;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, H);
  static constexpr int PRODUCTS = BF ? 1 : 3;       // tcgen05.mma per K step
};

// Parameter vectors are padded to 16 bytes so the mbarriers after them stay 8-byte aligned.
__host__ __device__ constexpr int padded_vec_floats(int n) { return (n + 3) & ~3; }

template <int H, bool BF>
constexpr uint32_t tile_smem_bytes(int n_vec_floats) {
  // ring (1024-aligned) + vectors + exchange buffers + barriers + alignment slack
  return TileGeom<H, BF>::RING_BYTES + (uint32_t)padded_vec_floats(n_vec_floats) * 4u + 256 + 1024;
}

// Launch geometry: dynamic shared memory of at least 120 KB, so that one CTA per SM runs (it owns
// the TMEM), and one persistent CTA per SM or per tile pair, whichever is fewer.
template <int H, bool BF>
constexpr uint32_t tile_launch_smem(int n_vec_floats) {
  return tile_smem_bytes<H, BF>(n_vec_floats) < 120u * 1024u ? 120u * 1024u : tile_smem_bytes<H, BF>(n_vec_floats);
}
inline int tile_grid(int n_tiles, int n_sm) {
  const int pairs = (n_tiles + 1) / 2;
  return pairs < n_sm ? pairs : n_sm;
}

// ----------------------------------------------------------------- kernel
template <TileKind KIND, int H, bool BF>
__global__ void __launch_bounds__(kThreads, 1) mlp_tile_kernel(const TileParams p) {
  using G = TileGeom<H, BF>;
  using SE = typename std::conditional<BF, __nv_bfloat16, float>::type;   // stored state element
  constexpr int NB = H / 8;                          // 8-column blocks per row
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* ring = smem;
  float* vecs = reinterpret_cast<float*>(smem + G::RING_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(vecs + padded_vec_floats(p.n_vec_floats));
  uint64_t* a_full = bars;                           // [2]  a slot's 8 worker warps published A
  uint64_t* d_full = bars + 2;                       // [2]  MMA of a slot's current job completed
  uint64_t* w_full = bars + 4;                       // [STAGES]  weight stage loaded
  uint64_t* w_empty = bars + 4 + G::STAGES;          // [STAGES]  both slots' MMAs on a stage completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 4 + 2 * G::STAGES);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* slot1_go = abort_flag + 1;          // slot 1 may start (edge kernels: the slots run out of phase)
  volatile int* cur_pair = abort_flag + 2;          // tile pair slot 0 is on (written only, see the worker loop)

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const bool resident = p.n_jobs <= G::STAGES;
  const int n_pairs = (p.n_tiles + 1) >> 1;

  for (int i = threadIdx.x; i < p.n_vec_floats; i += kThreads) vecs[i] = p.vecs[i];
  if (threadIdx.x == 0) {
    mbar_init(&a_full[0], 8); mbar_init(&a_full[1], 8);
    mbar_init(&d_full[0], 1); mbar_init(&d_full[1], 1);
    for (int s = 0; s < G::STAGES; ++s) { mbar_init(&w_full[s], 1); mbar_init(&w_empty[s], 2); }
    *abort_flag = 0;
    *slot1_go = 0;
    *cur_pair = -1;
    fence_mbar_init();
    if (resident) {                                    // the weights are constant: load them at once
      mbar_arrive_expect_tx(&w_full[0], (uint32_t)p.n_jobs * G::MAT_BYTES);
      for (int j = 0; j < p.n_jobs; ++j)
        bulk_g2s(ring + j * G::MAT_BYTES, p.wmats + (size_t)p.job_mat[j] * p.mat_bytes, G::MAT_BYTES, &w_full[0]);
    }
  }
  if (warp == 0) { tmem_alloc(tmem_slot, G::TMEM_COLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // Everything above (parameter vectors, barriers, tensor memory, the resident weights) depends on
  // no earlier kernel, so under a programmatic dependent launch it overlaps the previous kernel's
  // exit; from here on every thread may read what that kernel wrote.
  pdl_wait();

  if (warp < 4) {
    // Control warpgroup: hands registers to the worker warpgroups.
    setmaxnreg_dec<kControlRegs>();
      if (warp == 1) {
      // ------------------------------------------------ weight producer
      if (resident && lane == 0) drain_wait(&w_full[0], 0);     // the resident weights have landed
      if (!resident && lane == 0) {
        {
          uint32_t seq = 0;
          for (int pair = blockIdx.x; pair < n_pairs && !*abort_flag; pair += gridDim.x) {
            for (int j = 0; j < p.n_jobs; ++j, ++seq) {
              const int st = seq % G::STAGES;
              if (seq >= (uint32_t)G::STAGES &&
                  !bounded_wait(&w_empty[st], ((seq / G::STAGES) - 1) & 1, abort_flag, p.err)) break;
              mbar_arrive_expect_tx(&w_full[st], G::MAT_BYTES);
              bulk_g2s(ring + st * G::MAT_BYTES, p.wmats + (size_t)p.job_mat[j] * p.mat_bytes, G::MAT_BYTES, &w_full[st]);
            }
          }
          // before teardown, every copy this thread issued has landed (the last one per stage)
          const uint32_t first = seq > (uint32_t)G::STAGES ? seq - G::STAGES : 0u;
          for (uint32_t k = first; k < seq; ++k) drain_wait(&w_full[k % G::STAGES], (k / G::STAGES) & 1);
        }
      }
      __syncwarp();
    } else if (warp == 0) {
      // ------------------------------------------------ MMA issuer
      // The two slots advance independently: each has its own job cursor, and
      // the issuer serves whichever slot has published its next A operand.  In
      // streamed-weight mode both slots walk the same (pair, job) sequence of
      // ring stages; a stage is released after both slots' MMAs on it completed
      // (w_empty counts two commits; a slot without a tile in the last pair is
      // covered by a second commit of the other slot).
      if (lane == 0) {
        int pair_s[2] = {(int)blockIdx.x, (int)blockIdx.x};
        int job_s[2] = {0, 0};
        uint32_t seq_s[2] = {0, 0};
        uint32_t a_par[2] = {0, 0};
        bool act[2] = {2 * (int)blockIdx.x < p.n_tiles, 2 * (int)blockIdx.x + 1 < p.n_tiles};
        bool ok = true;
        if (resident) ok = bounded_wait(&w_full[0], 0, abort_flag, p.err);
        uint64_t t_last = global_timer_ns();
        uint32_t spins = 0;
        while (ok && (act[0] || act[1])) {
          bool progressed = false;
#pragma unroll
          for (int s = 0; s < 2; ++s) {
            if (!act[s]) continue;
            const int j = job_s[s];
            const int st = resident ? j : (int)(seq_s[s] % G::STAGES);
            if (!resident && !mbar_test_wait(&w_full[st], (seq_s[s] / G::STAGES) & 1)) continue;
            if (!mbar_test_wait(&a_full[s], a_par[s])) continue;
            a_par[s] ^= 1;
            GNN_TRACE_AT(0, 2 * (int)seq_s[s] + s * 256);
            tc_fence_after();
            const uint32_t wb = smem_u32(ring + st * G::MAT_BYTES);
            const uint32_t d = tmem_base + s * G::SLOT_COLS;
            const uint32_t ahi = d + H, alo = d + H + H / 2;
#pragma unroll 1
            for (int ks = 0; ks < H / 16; ++ks) {
              const uint32_t off = (ks >> 2) * (H * 128) + (ks & 3) * 32;
              const uint64_t bh = sdesc_kmajor_sw128(wb + off);
              const uint64_t bl = BF ? 0ull : sdesc_kmajor_sw128(wb + G::PART_BYTES + off);
              const uint32_t acc = (p.job_acc[j] || ks > 0) ? 1u : 0u;
              mma_bf16_ts(d, ahi + ks * 8, bh, G::IDESC, acc);
              if constexpr (!BF) {
                mma_bf16_ts(d, ahi + ks * 8, bl, G::IDESC, 1u);
                mma_bf16_ts(d, alo + ks * 8, bh, G::IDESC, 1u);
              }
            }
            mma_commit(&d_full[s]);
            GNN_TRACE_AT(0, 2 * (int)seq_s[s] + 1 + s * 256);
            if (!resident) {
              mma_commit(&w_empty[st]);
              if (s == 0 && 2 * pair_s[0] + 1 >= p.n_tiles) mma_commit(&w_empty[st]);   // slot 1 has no tile
            }
            seq_s[s]++;
            if (++job_s[s] == p.n_jobs) {
              job_s[s] = 0;
              pair_s[s] += gridDim.x;
              act[s] = 2 * pair_s[s] + s < p.n_tiles;
            }
            progressed = true;
          }
          if (progressed) {
            t_last = global_timer_ns();
            spins = 0;
          } else if ((++spins & 63u) == 0) {
            if (*abort_flag) break;
            if (global_timer_ns() - t_last > kWaitLimitNs) {
              atomicOr(p.err, DEV_ERR_TIMEOUT);
              *abort_flag = 1;
              break;
            }
          }
        }
        // before teardown (and the TMEM release), this thread's last MMAs of each slot have completed
        for (int s = 0; s < 2; ++s)
          if (seq_s[s] > 0) drain_wait(&d_full[s], (seq_s[s] - 1) & 1);
      }
      __syncwarp();
    }
  } else {
    // Worker warpgroups.
    setmaxnreg_inc<kWorkerRegs>();
    const int wq = warp - 4;                   // worker index 0..15
    const int slot = wq >> 3;
    const int ws = wq & 7;                     // warp index inside the slot
    const int quarter = warp & 3;              // TMEM lane quarter of this warp
    const int hq = (wq >> 2) & 1;
    const int lane_base = quarter * 32 + hq * 16;
    const int r0 = lane_base + (lane >> 2);    // first of the two rows inside the tile
    const int cq = 2 * (lane & 3);             // column offset inside a block
    const uint32_t lane_off = (uint32_t)lane_base << 16;
    const uint32_t slot_cols = tmem_base + slot * G::SLOT_COLS;
    const uint32_t d_addr = slot_cols + lane_off;
    const uint32_t ahi_addr = d_addr + H;
    const uint32_t alo_addr = d_addr + H + H / 2;
    uint32_t d_use = 0;
  #ifdef GNN_TRACE
    int tr_iter = 0;
    const int trow = (slot == 0 && ws == 2 && lane == 0) ? 0 : -1;
  #endif

    auto arrive_a = [&](int, uint32_t) {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[slot]);
    };
    auto wait_d = [&]() -> bool {              // never early-exits a tile
      const bool ok = bounded_wait(&d_full[slot], d_use & 1, abort_flag, p.err);
      d_use++;
      tc_fence_after();
      return ok;
    };
    auto quad_sum = [&](float x) {
      x += __shfl_xor_sync(0xffffffffu, x, 1);
      x += __shfl_xor_sync(0xffffffffu, x, 2);
      return x;
    };
    // Row data keep each thread's four values of a block pair (blocks 2bp and 2bp+1, columns
    // 2(t%4) and 2(t%4)+1 of each) together, so every row access is one 16-byte (fp32) or
    // 8-byte (bf16) vector:
    //   row-tiled state "T16" (e, h, a): (r, c) at ((r/128)*(H/16) + bp)*2048 + (r%128)*16 + x,
    //   row-major "RM16" (P_s, P_d, fp32): (r, c) at r*H + bp*16 + x,
    // with b = c/8, bp = b/2, x = 4*((c%8)/2) + 2*(b%2) + c%2.
    auto t16 = [&](const void* base, int row, int bp) -> const SE* {
      return static_cast<const SE*>(base) + (((size_t)(row >> 7) * (NB / 2) + bp) * 128 + (row & 127)) * 16 + 2 * cq;
    };
    auto ld_state = [&](const SE* a) -> float4 {
      if constexpr (BF) {
        const uint2 u = *reinterpret_cast<const uint2*>(a);
        const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
        const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
        return make_float4(lo.x, lo.y, hi.x, hi.y);
      } else {
        return *reinterpret_cast<const float4*>(a);
      }
    };
    auto st_state = [&](const SE* a, const float4& x) {
      if constexpr (BF) {
        *reinterpret_cast<uint2*>(const_cast<SE*>(a)) = make_uint2(pack_bf16x2(x.x, x.y), pack_bf16x2(x.z, x.w));
      } else {
        *reinterpret_cast<float4*>(const_cast<SE*>(a)) = x;
      }
    };
    auto rm16 = [&](const float* base, int row, int bp) -> const float4* {
      return reinterpret_cast<const float4*>(base + (size_t)row * H + bp * 16 + 2 * cq);
    };
    // Per-column parameter vectors (bias, gamma, beta, head weights, first-layer weight rows) are
    // stored by the host in block-pair order: column 8b + 2q + e of an H-vector at index
    // 16*(b/2) + 4q + 2*(b%2) + e.  The thread with q = lane % 4 reads its two columns of blocks
    // k and k+1 (k even) as one 16-byte vector, (.x, .y) for block k and (.z, .w) for block k+1,
    // and the four quad positions read 64 contiguous bytes (no bank conflict).
    const int qoff = (lane & 3) * 4;
    auto vq4 = [&](const float* x, int k) { return *reinterpret_cast<const float4*>(x + qoff + 8 * k); };
    // (row r0 quad values of blocks 2bp, 2bp+1) <-> v
    auto put4 = [&](float* v, int bp, int r, const float4& x) {
      v[8 * bp + 2 * r] = x.x; v[8 * bp + 2 * r + 1] = x.y; v[8 * bp + 4 + 2 * r] = x.z; v[8 * bp + 4 + 2 * r + 1] = x.w;
    };
    auto get4 = [&](const float* v, int bp, int r) {
      return make_float4(v[8 * bp + 2 * r], v[8 * bp + 2 * r + 1], v[8 * bp + 4 + 2 * r], v[8 * bp + 4 + 2 * r + 1]);
    };
    auto load_d = [&](float* v) {              // D of both rows, one TMEM round trip
#pragma unroll
      for (int c = 0; c < H; c += 64) tmem_ld_16x256b_x8(d_addr + c, v + c / 2);
      tmem_ld_wait();
    };
    // Blocks 4k..4k+3 of both rows (t[4b..4b+3] = block 4k+b: row 0 cols 2(t%4), +1; row 1 the same)
    // -> bf16 hi/lo A operand.  No wait: the caller ends a run of stores with tmem_st_wait().
    auto put_a_chunk = [&](int k, const float* t) {
      if constexpr (BF) {
        uint32_t hi[8];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          hi[2 * b] = pack_bf16x2(t[4 * b], t[4 * b + 1]);
          hi[2 * b + 1] = pack_bf16x2(t[4 * b + 2], t[4 * b + 3]);
        }
        tmem_st_16x128b_x4(ahi_addr + 16 * k, hi);
      } else {
        uint32_t hi[8], lo[8];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          split_bf16x2(t[4 * b], t[4 * b + 1], hi[2 * b], lo[2 * b]);
          split_bf16x2(t[4 * b + 2], t[4 * b + 3], hi[2 * b + 1], lo[2 * b + 1]);
        }
        tmem_st_16x128b_x4(ahi_addr + 16 * k, hi);
        tmem_st_16x128b_x4(alo_addr + 16 * k, lo);
      }
    };
    // both rows -> bf16 hi/lo A operand, four blocks per store pair (keeps the
    // temporaries at 16 registers next to the row data)
    auto put_a = [&](const float* v) {
#pragma unroll
      for (int k = 0; k < NB / 4; ++k) put_a_chunk(k, v + 16 * k);
      tmem_st_wait();
    };
    auto add_vec = [&](float* v, const float* b) {
#pragma unroll
      for (int k = 0; k < NB; k += 2) {
        const float4 t = vq4(b, k);
        v[4 * k] += t.x; v[4 * k + 1] += t.y; v[4 * k + 2] += t.x; v[4 * k + 3] += t.y;
        v[4 * k + 4] += t.z; v[4 * k + 5] += t.w; v[4 * k + 6] += t.z; v[4 * k + 7] += t.w;
      }
    };
    // LayerNorm (biased variance) + ReLU of both rows, in registers.  The host
    // centres every weight block and bias that feeds a LayerNorm (each output
    // row minus the mean over output rows), so the pre-activation reaching
    // here already has zero mean over the H features: the LayerNorm needs only
    // its variance (the subtraction of the mean is linear and sits in the MMA).
    auto ln_relu = [&](float* v, const float* gamma, const float* beta) {
      if constexpr (BF) {                      // bf16 weights are not centred: subtract the mean here
        float s0 = 0.f, s1 = 0.f;
#pragma unroll
        for (int k = 0; k < NB; ++k) { s0 += v[4 * k] + v[4 * k + 1]; s1 += v[4 * k + 2] + v[4 * k + 3]; }
        const float m0 = quad_sum(s0) * (1.0f / H), m1 = quad_sum(s1) * (1.0f / H);
#pragma unroll
        for (int k = 0; k < NB; ++k) { v[4 * k] -= m0; v[4 * k + 1] -= m0; v[4 * k + 2] -= m1; v[4 * k + 3] -= m1; }
      }
      float q0 = 0.f, q1 = 0.f;
#pragma unroll
      for (int k = 0; k < NB; ++k) {
        q0 = fmaf(v[4 * k], v[4 * k], fmaf(v[4 * k + 1], v[4 * k + 1], q0));
        q1 = fmaf(v[4 * k + 2], v[4 * k + 2], fmaf(v[4 * k + 3], v[4 * k + 3], q1));
      }
      const float i0 = rsqrtf(quad_sum(q0) * (1.0f / H) + p.eps);
      const float i1 = rsqrtf(quad_sum(q1) * (1.0f / H) + p.eps);
#pragma unroll
      for (int k = 0; k < NB; k += 2) {
        const float4 g = vq4(gamma, k), b = vq4(beta, k);
        v[4 * k] = fmaxf(fmaf(v[4 * k] * i0, g.x, b.x), 0.f);
        v[4 * k + 1] = fmaxf(fmaf(v[4 * k + 1] * i0, g.y, b.y), 0.f);
        v[4 * k + 2] = fmaxf(fmaf(v[4 * k + 2] * i1, g.x, b.x), 0.f);
        v[4 * k + 3] = fmaxf(fmaf(v[4 * k + 3] * i1, g.y, b.y), 0.f);
        v[4 * k + 4] = fmaxf(fmaf(v[4 * k + 4] * i0, g.z, b.z), 0.f);
        v[4 * k + 5] = fmaxf(fmaf(v[4 * k + 5] * i0, g.w, b.w), 0.f);
        v[4 * k + 6] = fmaxf(fmaf(v[4 * k + 6] * i1, g.z, b.z), 0.f);
        v[4 * k + 7] = fmaxf(fmaf(v[4 * k + 7] * i1, g.w, b.w), 0.f);
      }
    };
    // LayerNorm + ReLU of D + bias of both rows, streamed from tensor memory in
    // two passes (the squares for the variance, then the values), so that a
    // thread holds at most 32 columns at a time; emit(k, t) receives blocks
    // 4k..4k+3 in the put_a_chunk order.  D stays valid until the slot's next
    // MMA, which this thread has not released yet.
    auto ln_stream = [&](const float* bias, const float* gamma, const float* beta, auto&& emit) {
      float q0 = 0.f, q1 = 0.f, s0 = 0.f, s1 = 0.f;
      {
        float t[H / 2];
#pragma unroll
        for (int c = 0; c < H; c += 64) tmem_ld_16x256b_x8(d_addr + c, t + c / 2);
        tmem_ld_wait();
#pragma unroll
        for (int k = 0; k < NB; k += 2) {
          const float4 bb = vq4(bias, k);
          const float a0 = t[4 * k] + bb.x, a1 = t[4 * k + 1] + bb.y;
          const float c0 = t[4 * k + 2] + bb.x, c1 = t[4 * k + 3] + bb.y;
          const float a2 = t[4 * k + 4] + bb.z, a3 = t[4 * k + 5] + bb.w;
          const float c2 = t[4 * k + 6] + bb.z, c3 = t[4 * k + 7] + bb.w;
          q0 = fmaf(a0, a0, fmaf(a1, a1, fmaf(a2, a2, fmaf(a3, a3, q0))));
          q1 = fmaf(c0, c0, fmaf(c1, c1, fmaf(c2, c2, fmaf(c3, c3, q1))));
          if constexpr (BF) { s0 += (a0 + a1) + (a2 + a3); s1 += (c0 + c1) + (c2 + c3); }
        }
      }
      // fp32 model: the host centred the weights, the mean is zero.  bf16 model: one-pass moments.
      const float m0 = BF ? quad_sum(s0) * (1.0f / H) : 0.f;
      const float m1 = BF ? quad_sum(s1) * (1.0f / H) : 0.f;
      const float i0 = rsqrtf(fmaxf(quad_sum(q0) * (1.0f / H) - m0 * m0, 0.f) + p.eps);
      const float i1 = rsqrtf(fmaxf(quad_sum(q1) * (1.0f / H) - m1 * m1, 0.f) + p.eps);
      float t[2][16];                          // double buffer: chunk k+1 is read while chunk k is emitted
      tmem_ld_16x256b_x4(d_addr, t[0]);
      tmem_ld_wait();
#pragma unroll
      for (int k = 0; k < NB / 4; ++k) {
        if (k + 1 < NB / 4) tmem_ld_16x256b_x4(d_addr + 32 * (k + 1), t[(k + 1) & 1]);
        float* u = t[k & 1];
#pragma unroll
        for (int b = 0; b < 4; b += 2) {
          const int kb = 4 * k + b;                        // block index
          const float4 bb = vq4(bias, kb), g = vq4(gamma, kb), be = vq4(beta, kb);
          u[4 * b] = fmaxf(fmaf((u[4 * b] + bb.x - m0) * i0, g.x, be.x), 0.f);
          u[4 * b + 1] = fmaxf(fmaf((u[4 * b + 1] + bb.y - m0) * i0, g.y, be.y), 0.f);
          u[4 * b + 2] = fmaxf(fmaf((u[4 * b + 2] + bb.x - m1) * i1, g.x, be.x), 0.f);
          u[4 * b + 3] = fmaxf(fmaf((u[4 * b + 3] + bb.y - m1) * i1, g.y, be.y), 0.f);
          u[4 * b + 4] = fmaxf(fmaf((u[4 * b + 4] + bb.z - m0) * i0, g.z, be.z), 0.f);
          u[4 * b + 5] = fmaxf(fmaf((u[4 * b + 5] + bb.w - m0) * i0, g.w, be.w), 0.f);
          u[4 * b + 6] = fmaxf(fmaf((u[4 * b + 6] + bb.z - m1) * i1, g.z, be.z), 0.f);
          u[4 * b + 7] = fmaxf(fmaf((u[4 * b + 7] + bb.w - m1) * i1, g.w, be.w), 0.f);
        }
        emit(k, u);
        if (k + 1 < NB / 4) tmem_ld_wait();
      }
    };
    // blocks 4k..4k+3 of both rows -> row-tiled (T16) output rows
    auto store_t16_chunk = [&](void* base, int row0, bool ok0, bool ok1, int k, const float* t) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        if (ok0) st_state(t16(base, row0, 2 * k + j), get4(t, j, 0));
        if (ok1) st_state(t16(base, row0 + 8, 2 * k + j), get4(t, j, 1));
      }
    };
    auto load_t16 = [&](float* v, const void* base, int row0, bool ok0, bool ok1) {
      const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int bp = 0; bp < NB / 2; ++bp) {
        put4(v, bp, 0, ok0 ? ld_state(t16(base, row0, bp)) : z);
        put4(v, bp, 1, ok1 ? ld_state(t16(base, row0 + 8, bp)) : z);
      }
    };
    auto store_t16 = [&](void* base, int row0, bool ok0, bool ok1, const float* v) {
#pragma unroll
      for (int bp = 0; bp < NB / 2; ++bp) {
        if (ok0) st_state(t16(base, row0, bp), get4(v, bp, 0));
        if (ok1) st_state(t16(base, row0 + 8, bp), get4(v, bp, 1));
      }
    };
    // D (+ bias) of both rows streamed to a row-major output, 4 blocks per TMEM round trip.
    auto stream_d = [&](float* base, int row0, bool ok0, bool ok1, const float* bias) {
#pragma unroll
      for (int c = 0; c < H; c += 32) {
        float t[16];
        tmem_ld_16x256b_x4(d_addr + c, t);
        tmem_ld_wait();
        if (bias) {
#pragma unroll
          for (int k = 0; k < 4; k += 2) {
            const float4 bb = vq4(bias, c / 8 + k);
            t[4 * k] += bb.x; t[4 * k + 1] += bb.y; t[4 * k + 2] += bb.x; t[4 * k + 3] += bb.y;
            t[4 * k + 4] += bb.z; t[4 * k + 5] += bb.w; t[4 * k + 6] += bb.z; t[4 * k + 7] += bb.w;
          }
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) {                    // block pairs of this 32-column chunk
          const int bp = c / 16 + k;
          if (ok0) *const_cast<float4*>(rm16(base, row0, bp)) = get4(t, k, 0);
          if (ok1) *const_cast<float4*>(rm16(base, row0 + 8, bp)) = get4(t, k, 1);
        }
      }
    };

    const int L = p.n_layers;
    bool ok = true;
    uint32_t seq = 0;                          // this slot's job sequence number
    for (int pair = blockIdx.x; ok && pair < n_pairs; pair += gridDim.x) {
      const int tile = 2 * pair + slot;
      if (tile >= p.n_tiles) break;
      const int row0 = tile * kTileRows + r0, row1 = row0 + 8;
      const bool ok0 = row0 < p.n_rows, ok1 = row1 < p.n_rows;
      float v[4 * NB];
      int j = 0;                               // job index inside the tile
      auto next_job = [&]() { ++j; ++seq; };
      auto wait_job = [&]() { ok &= wait_d(); };

      if constexpr (KIND == TileKind::EdgeUpdate || KIND == TileKind::Classifier) {
        // vec layout: [gamma1, beta1, (b_l, gamma_l, beta_l) for l = 2..L, (w_o, b_o)]
        // The two slots run out of phase: slot 1 starts once slot 0 has released the last MMA of
        // its first tile, so that one slot's tile change (store, next loads) overlaps the other
        // slot's MMAs instead of leaving the tensor core idle.  Bounded: it starts anyway after
        // the wait limit.
        if (slot == 1 && pair == (int)blockIdx.x) {
          const uint64_t t0 = global_timer_ns();
          for (uint32_t it = 0; *slot1_go == 0; ++it) {
            if (*abort_flag || ((it & 255u) == 255u && global_timer_ns() - t0 > kWaitLimitNs)) break;
            __nanosleep(64);
          }
        }
        // Edge update: slot 0 records its tile pair.  Nothing reads the word; the store stays
        // because without it ptxas allocates the fp32 edge update's worker registers differently
        // and spills 28 B (measured: 0.391 -> 0.404 ms per launch).  The classifier is faster
        // without it (0.384 -> 0.373 ms).
        if (KIND == TileKind::EdgeUpdate && slot == 0 && ws == 0 && lane == 0) *cur_pair = pair;
        auto release_slot1 = [&]() {
          if (slot == 0 && pair == (int)blockIdx.x && j == L && ws == 0 && lane == 0) *slot1_go = 1;
        };
        GNN_TRACE_W(0);
        const int s0 = ok0 ? p.src_sorted[row0] : 0, d0 = ok0 ? p.dst_sorted[row0] : 0;
        const int s1 = ok1 ? p.src_sorted[row1] : 0, d1 = ok1 ? p.dst_sorted[row1] : 0;
        // classifier: where each row's score goes (input order) and, in the sign bit, whether an
        // endpoint was out of range; read now so that the score store ending the tile waits on no
        // load (measured: 0.4205 -> 0.4095 ms per launch on the full event)
        int out0 = 0, out1 = 0;
        if constexpr (KIND == TileKind::Classifier) {
          if (ok0 && (lane & 3) == 0) out0 = p.perm[row0] | (p.key_sorted[row0] < p.n_nodes ? 0 : INT_MIN);
          if (ok1 && (lane & 3) == 0) out1 = p.perm[row1] | (p.key_sorted[row1] < p.n_nodes ? 0 : INT_MIN);
        }
        load_t16(v, p.e, row0, ok0, ok1);
        GNN_TRACE_W(1);
        put_a(v);
        arrive_a(j, seq); next_job(); release_slot1();                     // job: D = e * W_e^T
        GNN_TRACE_W(2);
        // layer-1 terms of the endpoints, loaded while the MMA runs: P_s[src] + P_d[dst] (P_d carries
        // b1).  P_s rows go straight into v; P_d rows follow two block pairs at a time, so at most
        // 16 registers of loads are in flight next to the row data.
#pragma unroll
        for (int bp = 0; bp < NB / 2; ++bp) {
          put4(v, bp, 0, *rm16(p.ps, s0, bp));
          put4(v, bp, 1, *rm16(p.ps, s1, bp));
        }
#pragma unroll
        for (int g = 0; g < NB / 2; g += 2) {
          float4 b[4];
#pragma unroll
          for (int k = 0; k < 2; ++k) { b[2 * k] = *rm16(p.pd, d0, g + k); b[2 * k + 1] = *rm16(p.pd, d1, g + k); }
#pragma unroll
          for (int k = 0; k < 2; ++k) {
            const float4 x0 = get4(v, g + k, 0), x1 = get4(v, g + k, 1);
            const float4& y0 = b[2 * k];
            const float4& y1 = b[2 * k + 1];
            put4(v, g + k, 0, make_float4(x0.x + y0.x, x0.y + y0.y, x0.z + y0.z, x0.w + y0.w));
            put4(v, g + k, 1, make_float4(x1.x + y1.x, x1.y + y1.y, x1.z + y1.z, x1.w + y1.w));
          }
        }
        GNN_TRACE_W(3);
        wait_job();
        GNN_TRACE_W(5);
#pragma unroll
        for (int c = 0; c < H; c += 32) {                 // v += D, 32 columns per TMEM round trip
          float t[16];
          tmem_ld_16x256b_x4(d_addr + c, t);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) v[c / 2 + i] += t[i];
        }
        ln_relu(v, vecs, vecs + H);
        put_a(v);
        arrive_a(j, seq); next_job(); release_slot1();
        GNN_TRACE_W(6);
        for (int l = 2; l <= L; ++l) {
          wait_job();
          GNN_TRACE_W(5 + 2 * (l - 1));
          if ((KIND == TileKind::EdgeUpdate || (KIND == TileKind::Classifier && !BF)) && l == 2 && ws == 0 &&
              lane == 0) {
            // Warm L2 with this slot's next edge-state tile, a few microseconds before its load
            // (bulk prefetch: the copy engine, not the SM's load path).  Measured on the full
            // event: edge update 0.484 -> 0.395 ms per launch; issued after layer 1 (0.420) or
            // layer 3 (0.412) it helps less.  Classifier: 0.376 ms against 0.394 without any
            // prefetch and 0.416 with a warp prefetching the next pair's tiles and gathered rows;
            // the bf16 classifier is fastest without prefetch (0.331, 0.342 with this one).
            const int nt = tile + 2 * (int)gridDim.x;
            if (nt < p.n_tiles)
              prefetch_l2_bulk(static_cast<const SE*>(p.e) + (size_t)nt * kTileRows * H, kTileRows * H * sizeof(SE));
          }
          load_d(v);
          const float* vb = vecs + (2 + 3 * (l - 2)) * H;
          add_vec(v, vb);
          ln_relu(v, vb + H, vb + 2 * H);
          if (l < L) { put_a(v); arrive_a(j, seq); next_job(); release_slot1(); }
          GNN_TRACE_W(6 + 2 * (l - 1));
        }
        if constexpr (KIND == TileKind::EdgeUpdate) {
          store_t16(p.e, row0, ok && ok0, ok && ok1, v);
          GNN_TRACE_W(11);
        } else {
          const float* wo = vecs + (2 + 3 * (L - 1)) * H;
          if constexpr (BF) {                  // the head's input is a bf16 activation
#pragma unroll
            for (int i = 0; i < 4 * NB; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
          }
          float z0 = 0.f, z1 = 0.f;
#pragma unroll
          for (int k = 0; k < NB; k += 2) {
            const float4 w = vq4(wo, k);
            z0 = fmaf(v[4 * k], w.x, fmaf(v[4 * k + 1], w.y, fmaf(v[4 * k + 4], w.z, fmaf(v[4 * k + 5], w.w, z0))));
            z1 = fmaf(v[4 * k + 2], w.x, fmaf(v[4 * k + 3], w.y, fmaf(v[4 * k + 6], w.z, fmaf(v[4 * k + 7], w.w, z1))));
          }
          z0 = quad_sum(z0) + wo[H];
          z1 = quad_sum(z1) + wo[H];
          if (ok && (lane & 3) == 0) {
            const float nan = __int_as_float(0x7fc00000);
            if (ok0) p.scores[out0 & INT_MAX] = out0 >= 0 ? 1.0f / (1.0f + __expf(-z0)) : nan;
            if (ok1) p.scores[out1 & INT_MAX] = out1 >= 0 ? 1.0f / (1.0f + __expf(-z1)) : nan;
          }
        }
      } else if constexpr (KIND == TileKind::EdgeEncoder) {
        // vec layout: [W1^T (2 x H), b1, gamma1, beta1, (b_l, gamma_l, beta_l) for l = 2..L]
        float f[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int row = r ? row1 : row0;
          if (r ? ok1 : ok0) {
            const int s = p.src_sorted[row], d = p.dst_sorted[row];
            const float* xs = p.x + (size_t)s * p.x_stride;
            const float* xd = p.x + (size_t)d * p.x_stride;
            f[r][0] = xd[0] - xs[0];
            float dphi = xd[1] - xs[1];
            if (dphi > 1.0f) dphi -= 2.0f;
            if (dphi <= -1.0f) dphi += 2.0f;
            f[r][1] = dphi;
          }
        }
        const float* vb = vecs + 2 * H;
#pragma unroll
        for (int k = 0; k < NB; k += 2) {
          const float4 w0 = vq4(vecs, k), w1 = vq4(vecs + H, k);
          v[4 * k] = fmaf(w1.x, f[0][1], w0.x * f[0][0]);
          v[4 * k + 1] = fmaf(w1.y, f[0][1], w0.y * f[0][0]);
          v[4 * k + 2] = fmaf(w1.x, f[1][1], w0.x * f[1][0]);
          v[4 * k + 3] = fmaf(w1.y, f[1][1], w0.y * f[1][0]);
          v[4 * k + 4] = fmaf(w1.z, f[0][1], w0.z * f[0][0]);
          v[4 * k + 5] = fmaf(w1.w, f[0][1], w0.w * f[0][0]);
          v[4 * k + 6] = fmaf(w1.z, f[1][1], w0.z * f[1][0]);
          v[4 * k + 7] = fmaf(w1.w, f[1][1], w0.w * f[1][0]);
        }
        add_vec(v, vb);
        ln_relu(v, vb + H, vb + 2 * H);
        put_a(v);
        arrive_a(j, seq); next_job();
        // Deeper layers: the fp32 model streams its epilogues, the bf16 model keeps the row in
        // registers (measured per launch, streamed / register form: fp32 0.285 / 0.293 ms, bf16
        // 0.232 / 0.219 ms).
        for (int l = 2; l < L; ++l) {
          wait_job();
          const float* vl = vb + 3 * (l - 1) * H;
          if constexpr (BF) {
            load_d(v);
            add_vec(v, vl);
            ln_relu(v, vl + H, vl + 2 * H);
            put_a(v);
          } else {
            ln_stream(vl, vl + H, vl + 2 * H, [&](int k, const float* t) { put_a_chunk(k, t); });
            tmem_st_wait();
          }
          arrive_a(j, seq); next_job();
        }
        wait_job();
        {
          const float* vl = vb + 3 * (L - 1) * H;
          const bool w0 = ok && ok0, w1 = ok && ok1;
          if constexpr (BF) {
            load_d(v);
            add_vec(v, vl);
            ln_relu(v, vl + H, vl + 2 * H);
            store_t16(p.e, row0, w0, w1, v);
          } else {
            ln_stream(vl, vl + H, vl + 2 * H, [&](int k, const float* t) { store_t16_chunk(p.e, row0, w0, w1, k, t); });
          }
        }
      } else if constexpr (KIND == TileKind::Embed) {
        // vec layout: [W1^T (F_n x H), (b_l, gamma_l, beta_l) for l = 1..L, W_out rows (D x H), b_out (D)]
        // L hidden layers (layer 1 on CUDA cores), then the D outputs on CUDA cores, L2-normalised.
#pragma unroll
        for (int i = 0; i < 4 * NB; ++i) v[i] = 0.f;
        for (int k = 0; k < p.n_feat; ++k) {
          const float x0 = ok0 ? p.x[(size_t)row0 * p.x_stride + k] : 0.f;
          const float x1 = ok1 ? p.x[(size_t)row1 * p.x_stride + k] : 0.f;
#pragma unroll
          for (int b = 0; b < NB; b += 2) {
            const float4 w = vq4(vecs + k * H, b);
            v[4 * b] = fmaf(w.x, x0, v[4 * b]); v[4 * b + 1] = fmaf(w.y, x0, v[4 * b + 1]);
            v[4 * b + 2] = fmaf(w.x, x1, v[4 * b + 2]); v[4 * b + 3] = fmaf(w.y, x1, v[4 * b + 3]);
            v[4 * b + 4] = fmaf(w.z, x0, v[4 * b + 4]); v[4 * b + 5] = fmaf(w.w, x0, v[4 * b + 5]);
            v[4 * b + 6] = fmaf(w.z, x1, v[4 * b + 6]); v[4 * b + 7] = fmaf(w.w, x1, v[4 * b + 7]);
          }
        }
        const float* vb = vecs + p.n_feat * H;
        add_vec(v, vb);
        ln_relu(v, vb + H, vb + 2 * H);
        for (int l = 2; l <= L; ++l) {
          put_a(v);
          arrive_a(j, seq); next_job();
          wait_job();
          load_d(v);
          const float* vl = vb + 3 * (l - 1) * H;
          add_vec(v, vl);
          ln_relu(v, vl + H, vl + 2 * H);
        }
        if constexpr (BF) {                  // the projection's input is a bf16 activation
#pragma unroll
          for (int i = 0; i < 4 * NB; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
        }
        const float* wout = vb + 3 * L * H;
        float y0[kMaxEmbedDim], y1[kMaxEmbedDim];
        float n0 = 0.f, n1 = 0.f;
        for (int d = 0; d < p.emb_dim; ++d) {
          float z0 = 0.f, z1 = 0.f;
#pragma unroll
          for (int k = 0; k < NB; k += 2) {
            const float4 w = vq4(wout + d * H, k);
            z0 = fmaf(v[4 * k], w.x, fmaf(v[4 * k + 1], w.y, fmaf(v[4 * k + 4], w.z, fmaf(v[4 * k + 5], w.w, z0))));
            z1 = fmaf(v[4 * k + 2], w.x, fmaf(v[4 * k + 3], w.y, fmaf(v[4 * k + 6], w.z, fmaf(v[4 * k + 7], w.w, z1))));
          }
          const float bo = wout[p.emb_dim * H + d];
          z0 = quad_sum(z0) + bo;
          z1 = quad_sum(z1) + bo;
#pragma unroll
          for (int i = 0; i < kMaxEmbedDim; ++i)
            if (i == d) { y0[i] = z0; y1[i] = z1; }
          n0 = fmaf(z0, z0, n0);
          n1 = fmaf(z1, z1, n1);
        }
        const float i0 = n0 > 0.f ? rsqrtf(n0) : 0.f, i1 = n1 > 0.f ? rsqrtf(n1) : 0.f;
        if (ok && (lane & 3) == 0) {
#pragma unroll
          for (int i = 0; i < kMaxEmbedDim; ++i) {
            if (i < p.emb_dim) {
              if (ok0) p.emb[(size_t)row0 * p.emb_dim + i] = y0[i] * i0;
              if (ok1) p.emb[(size_t)row1 * p.emb_dim + i] = y1[i] * i1;
            }
          }
        }
      } else if constexpr (KIND == TileKind::Filter) {
        // vec layout: [W1^T (2 F_n x H), b1, gamma1, beta1, (b_l, gamma_l, beta_l) for l = 2..L, (w_o, b_o)]
        // Layer 1 on CUDA cores from the raw features of both endpoints, [x_src, x_dst].
        bool valid[2] = {false, false};
        int sv[2] = {0, 0}, dv[2] = {0, 0};
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int row = r ? row1 : row0;
          if (r ? ok1 : ok0) {
            const int s = p.ei_in[row], d = p.ei_in[(size_t)p.n_rows + row];
            valid[r] = s >= 0 && s < p.n_nodes && d >= 0 && d < p.n_nodes;
            sv[r] = valid[r] ? s : 0;
            dv[r] = valid[r] ? d : 0;
          }
        }
#pragma unroll
        for (int i = 0; i < 4 * NB; ++i) v[i] = 0.f;
        for (int k = 0; k < 2 * p.n_feat; ++k) {
          const int node0 = k < p.n_feat ? sv[0] : dv[0], node1 = k < p.n_feat ? sv[1] : dv[1];
          const int col = k < p.n_feat ? k : k - p.n_feat;
          const float x0 = valid[0] ? p.x[(size_t)node0 * p.x_stride + col] : 0.f;
          const float x1 = valid[1] ? p.x[(size_t)node1 * p.x_stride + col] : 0.f;
#pragma unroll
          for (int b = 0; b < NB; b += 2) {
            const float4 w = vq4(vecs + k * H, b);
            v[4 * b] = fmaf(w.x, x0, v[4 * b]); v[4 * b + 1] = fmaf(w.y, x0, v[4 * b + 1]);
            v[4 * b + 2] = fmaf(w.x, x1, v[4 * b + 2]); v[4 * b + 3] = fmaf(w.y, x1, v[4 * b + 3]);
            v[4 * b + 4] = fmaf(w.z, x0, v[4 * b + 4]); v[4 * b + 5] = fmaf(w.w, x0, v[4 * b + 5]);
            v[4 * b + 6] = fmaf(w.z, x1, v[4 * b + 6]); v[4 * b + 7] = fmaf(w.w, x1, v[4 * b + 7]);
          }
        }
        const float* vb = vecs + 2 * p.n_feat * H;
        add_vec(v, vb);
        ln_relu(v, vb + H, vb + 2 * H);
        for (int l = 2; l <= L; ++l) {
          put_a(v);
          arrive_a(j, seq); next_job();
          wait_job();
          load_d(v);
          const float* vl = vb + 3 * (l - 1) * H;
          add_vec(v, vl);
          ln_relu(v, vl + H, vl + 2 * H);
        }
        const float* wo = vb + 3 * L * H;
        if constexpr (BF) {                  // the head's input is a bf16 activation
#pragma unroll
          for (int i = 0; i < 4 * NB; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
        }
        float z0 = 0.f, z1 = 0.f;
#pragma unroll
        for (int k = 0; k < NB; k += 2) {
          const float4 w = vq4(wo, k);
          z0 = fmaf(v[4 * k], w.x, fmaf(v[4 * k + 1], w.y, fmaf(v[4 * k + 4], w.z, fmaf(v[4 * k + 5], w.w, z0))));
          z1 = fmaf(v[4 * k + 2], w.x, fmaf(v[4 * k + 3], w.y, fmaf(v[4 * k + 6], w.z, fmaf(v[4 * k + 7], w.w, z1))));
        }
        z0 = quad_sum(z0) + wo[H];
        z1 = quad_sum(z1) + wo[H];
        if (ok && (lane & 3) == 0) {
          const float nan = __int_as_float(0x7fc00000);
          if (ok0) p.scores[row0] = valid[0] ? 1.0f / (1.0f + __expf(-z0)) : nan;
          if (ok1) p.scores[row1] = valid[1] ? 1.0f / (1.0f + __expf(-z1)) : nan;
          if ((ok0 && !valid[0]) || (ok1 && !valid[1])) atomicOr(p.err, DEV_ERR_INDEX_RANGE);
        }
      } else {
        // NodeEncoder / NodeUpdate.
        // vec layout: [W1^T (n_feat x H) if encoder], (b_l, gamma_l, beta_l) for l = 1..L, b1_edge
        const float* vb = vecs + (KIND == TileKind::NodeEncoder ? p.n_feat * H : 0);
        int l0;
        if constexpr (KIND == TileKind::NodeEncoder) {
#pragma unroll
          for (int i = 0; i < 4 * NB; ++i) v[i] = 0.f;
          for (int k = 0; k < p.n_feat; ++k) {            // layer 1 on CUDA cores
            const float x0 = ok0 ? p.x[(size_t)row0 * p.x_stride + k] : 0.f;
            const float x1 = ok1 ? p.x[(size_t)row1 * p.x_stride + k] : 0.f;
#pragma unroll
            for (int b = 0; b < NB; b += 2) {
              const float4 w = vq4(vecs + k * H, b);
              v[4 * b] = fmaf(w.x, x0, v[4 * b]); v[4 * b + 1] = fmaf(w.y, x0, v[4 * b + 1]);
              v[4 * b + 2] = fmaf(w.x, x1, v[4 * b + 2]); v[4 * b + 3] = fmaf(w.y, x1, v[4 * b + 3]);
              v[4 * b + 4] = fmaf(w.z, x0, v[4 * b + 4]); v[4 * b + 5] = fmaf(w.w, x0, v[4 * b + 5]);
              v[4 * b + 6] = fmaf(w.z, x1, v[4 * b + 6]); v[4 * b + 7] = fmaf(w.w, x1, v[4 * b + 7]);
            }
          }
          add_vec(v, vb);
          ln_relu(v, vb + H, vb + 2 * H);
          put_a(v);
          arrive_a(j, seq); next_job();
          l0 = 2;
        } else {
          GNN_TRACE_W(0);
          load_t16(v, p.h, row0, ok0, ok1);
          put_a(v);
          arrive_a(j, seq); next_job();                   // job: D = h * W_h^T
          GNN_TRACE_W(1);
          if (KIND == TileKind::NodeUpdate && ws == 0 && lane == 0)   // this tile's aggregate rows
            prefetch_l2_bulk(static_cast<const SE*>(p.agg) + (size_t)tile * kTileRows * H, kTileRows * H * sizeof(SE));
          // The aggregate rows are loaded only after the first job completed: a burst of global
          // loads from a slot's warps while its MMAs run slows those MMAs several-fold (the loads
          // compete with the tensor core's operand reads in the SM's memory pipeline).
          GNN_TRACE_W(2);
          wait_job();                                     // A free again
          GNN_TRACE_W(3);
          load_t16(v, p.agg, row0, ok0, ok1);              // a_j, summed by the aggregation kernel
          put_a(v);
          arrive_a(j, seq); next_job();                   // job: D += a * W_a^T
          GNN_TRACE_W(4);
          l0 = 1;
        }
        for (int l = l0; l < L; ++l) {
          wait_job();
          GNN_TRACE_W(3 + 2 * l);
          const float* vl = vb + 3 * (l - 1) * H;
          ln_stream(vl, vl + H, vl + 2 * H, [&](int k, const float* t) { put_a_chunk(k, t); });
          tmem_st_wait();
          arrive_a(j, seq); next_job();                   // next layer
          GNN_TRACE_W(4 + 2 * l);
        }
        if (l0 <= L) {                                    // last layer: new node state, and A for the P_s job
          wait_job();
          if (KIND == TileKind::NodeUpdate && ws == 0 && lane == 0) {
            // This slot's next h tile, ~10 us before its load.  Measured on the full event with the
            // aggregate prefetch above: 0.223 -> 0.196 ms per launch; both tiles prefetched a whole
            // tile ahead made it slower (0.248), prefetching later helps less.
            const int nt = tile + 2 * (int)gridDim.x;
            if (nt < p.n_tiles)
              prefetch_l2_bulk(static_cast<const SE*>(p.h) + (size_t)nt * kTileRows * H, kTileRows * H * sizeof(SE));
          }
          GNN_TRACE_W(3 + 2 * L);
          const float* vl = vb + 3 * (L - 1) * H;
          const bool w0 = ok && ok0, w1 = ok && ok1;
          ln_stream(vl, vl + H, vl + 2 * H, [&](int k, const float* t) {
            store_t16_chunk(p.h, row0, w0, w1, k, t);
            put_a_chunk(k, t);
          });
          tmem_st_wait();
          arrive_a(j, seq); next_job();                   // the P_s job
        }
        GNN_TRACE_W(11);
        wait_job();                                       // P_s = W_s h (no bias)
        GNN_TRACE_W(12);
        stream_d(p.ps, row0, ok && ok0, ok && ok1, nullptr);
        tmem_ld_wait();
        arrive_a(j, seq); next_job();                     // D read; A (= h) unchanged -> P_d job
        GNN_TRACE_W(13);
        wait_job();                                       // P_d = W_d h + b1 (edge-side bias)
        GNN_TRACE_W(14);
        stream_d(p.pd, row0, ok && ok0, ok && ok1, vb + 3 * L * H);
        GNN_TRACE_W(15);
      }
      if (!ok) break;                          // leave only between tiles
  #ifdef GNN_TRACE
      ++tr_iter;
  #endif
    }
    __syncwarp();
  }

  // teardown: every warp reaches this point (waits are bounded)
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, G::TMEM_COLS);
  }
}

// a_j = sum of the messages m_ij of the edges into node j (CSR segment of j,
// summed in slot order from zero, no atomics: deterministic, and identical for
// a node whether its event is scored alone or in a batch).  One warp serves one
// node (half a warp when H = 64): lane 4*bp + q owns the 16-byte vector q of
// block pair bp (row-tiled T16 layout of the tile kernels), so all lanes of a
// node run the same number of steps whatever the degree distribution, and
// every message row is read in whole 64-byte pieces.  Blocks take the nodes
// from the last one down: the edge update writes the messages in CSR (that is,
// destination) order and finishes with the highest tiles, which are then still
// in L2 when the first blocks here read them.
template <int H>
constexpr int agg_nodes_per_block() { return 256 / (H / 4); }

template <int H, bool BF>
__global__ void __launch_bounds__(256) aggregate_kernel(const void* __restrict__ e_, const int* __restrict__ rowptr,
                                                        int n_nodes, void* __restrict__ agg_) {
  using SE = typename std::conditional<BF, __nv_bfloat16, float>::type;
  constexpr int NBP = H / 16;
  constexpr int LPN = H / 4;                         // lanes per node
  const SE* e = static_cast<const SE*>(e_);
  SE* agg = static_cast<SE*>(agg_);
  pdl_wait();
  const int li = threadIdx.x % LPN;
  const int bp = li >> 2, q = li & 3;
  const int j = n_nodes - 1 - (blockIdx.x * agg_nodes_per_block<H>() + (int)threadIdx.x / LPN);
  if (j < 0) return;
  const int k0 = rowptr[j], k1 = rowptr[j + 1];
  auto at = [&](int k) -> float4 {
    const SE* a = e + (((size_t)(k >> 7) * NBP + bp) * 128 + (k & 127)) * 16 + 4 * q;
    if constexpr (BF) {
      const uint2 u = __ldcs(reinterpret_cast<const uint2*>(a));
      const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.x));
      const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&u.y));
      return make_float4(lo.x, lo.y, hi.x, hi.y);
    } else {
      return __ldcs(reinterpret_cast<const float4*>(a));
    }
  };
  float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
  int k = k0;
  for (; k + 4 <= k1; k += 4) {
    const float4 x0 = at(k), x1 = at(k + 1), x2 = at(k + 2), x3 = at(k + 3);
    a.x += x0.x; a.y += x0.y; a.z += x0.z; a.w += x0.w;
    a.x += x1.x; a.y += x1.y; a.z += x1.z; a.w += x1.w;
    a.x += x2.x; a.y += x2.y; a.z += x2.z; a.w += x2.w;
    a.x += x3.x; a.y += x3.y; a.z += x3.z; a.w += x3.w;
  }
  for (; k < k1; ++k) {
    const float4 x = at(k);
    a.x += x.x; a.y += x.y; a.z += x.z; a.w += x.w;
  }
  SE* out = agg + (((size_t)(j >> 7) * NBP + bp) * 128 + (j & 127)) * 16 + 4 * q;
  if constexpr (BF) {                                // the aggregate is a bf16 activation
    *reinterpret_cast<uint2*>(out) = make_uint2(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w));
  } else {
    *reinterpret_cast<float4*>(out) = a;
  }
}

}  // namespace gnn
