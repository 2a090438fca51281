// Fused MLP-tile kernels of the interaction network (tcgen05 / TMEM, sm_103a).
//
// One persistent CTA per SM walks 128-row tiles (edges in destination-sorted
// CSR order, or nodes).  Each tile runs a fixed program of "jobs": a job is one
// Linear layer D = A * W^T executed on the 5th-generation tensor cores with
// the activation tile A in tensor memory and the weight W in shared memory,
// followed by an epilogue in registers (bias or gathered projections,
// LayerNorm, ReLU) that writes the next layer's A back into tensor memory.
//
// Precision: fp32 model, every product evaluated as hi*hi + hi*lo + lo*hi of
// bf16 splits (v = hi + lo, both bf16) with fp32 accumulation, which keeps the
// relative product error near 2^-16.
//
// Roles (576 threads = 18 warps):
//   warp 0      : MMA issuer (one elected lane)
//   warp 1      : weight producer (bulk copies into the smem weight ring)
//   warps 2..17 : 16 row-worker warps = 2 slots x 2 column halves x 4 lane
//                 quarters.  Slot s works on tiles 2p+s of tile pair p, so the
//                 tensor core alternates between the two slots (ping-pong) and
//                 one slot's epilogue overlaps the other slot's MMAs.
// Each row of a tile is owned by two threads (column halves); LayerNorm
// statistics are combined through a small shared-memory exchange.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>
#include "ptx.cuh"

namespace gnn {

enum class TileKind : int {
  NodeEncoder = 0,     // x -> h0 (layer 1 on CUDA cores), then P_s, P_d projections
  EdgeEncoder = 1,     // (dr, dphi) -> e0 (layer 1 on CUDA cores)
  EdgeUpdate  = 2,     // e <- MLP_edge([h_src, h_dst, e]) via e*W_e + P_s[src] + P_d[dst]
  NodeUpdate  = 3,     // h <- MLP_node([h, sum of incoming e]); then P_s, P_d of new h
  Classifier  = 4,     // score = sigmoid(w_o . MLP_cls([h_src, h_dst, e]) + b_o)
};

constexpr int kThreads = 576;
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
  float* e;                   // [E, H] edge state, CSR order (updated in place)
  float* h;                   // [N, H] node state
  float* ps;                  // [N, H] projections W_s h
  float* pd;                  // [N, H] projections W_d h + b1
  float* scores;              // [E] input order
  uint32_t* err;              // device error word
};

template <int H>
struct TileGeom {
  static constexpr int HH = H / 2;                  // columns per worker thread
  static constexpr int SLOT_COLS = 2 * H;           // D (H cols) + A_hi (H/2) + A_lo (H/2)
  static constexpr int TMEM_COLS = 2 * SLOT_COLS;   // two slots: 256 (H=64) or 512 (H=128)
  static constexpr uint32_t PART_BYTES = H * H * 2; // one bf16 H x H matrix part
  static constexpr uint32_t MAT_BYTES = 2 * PART_BYTES;
  static constexpr int STAGES = (H == 128) ? 3 : 8; // weight ring depth (matrices)
  static constexpr uint32_t RING_BYTES = STAGES * MAT_BYTES;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, H);
};

// Parameter vectors are padded to 16 bytes so the mbarriers after them stay 8-byte aligned.
__host__ __device__ constexpr int padded_vec_floats(int n) { return (n + 3) & ~3; }

template <int H>
constexpr uint32_t tile_smem_bytes(int n_vec_floats) {
  // ring (1024-aligned) + vectors + exchange buffers + barriers + alignment slack
  return TileGeom<H>::RING_BYTES + (uint32_t)padded_vec_floats(n_vec_floats) * 4u + 2 * 2 * 2 * 128 * 4 +
         256 + 1024;
}

// ----------------------------------------------------------------- kernel
template <TileKind KIND, int H>
__global__ void __launch_bounds__(kThreads, 1) mlp_tile_kernel(const TileParams p) {
  using G = TileGeom<H>;
  constexpr int HH = G::HH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* ring = smem;
  float* vecs = reinterpret_cast<float*>(smem + G::RING_BYTES);
  float* red = vecs + padded_vec_floats(p.n_vec_floats);    // [2 slot][2 buf][2 half][128]
  uint64_t* bars = reinterpret_cast<uint64_t*>(red + 2 * 2 * 2 * 128);
  uint64_t* a_full = bars;          // [2]
  uint64_t* d_full = bars + 2;      // [2]
  uint64_t* w_full = bars + 4;      // [STAGES]
  uint64_t* w_empty = bars + 4 + G::STAGES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 4 + 2 * G::STAGES);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const bool resident = p.n_jobs <= G::STAGES;

  for (int i = threadIdx.x; i < p.n_vec_floats; i += kThreads) vecs[i] = p.vecs[i];
  if (threadIdx.x == 0) {
    mbar_init(&a_full[0], 8); mbar_init(&a_full[1], 8);
    mbar_init(&d_full[0], 1); mbar_init(&d_full[1], 1);
    for (int s = 0; s < G::STAGES; ++s) { mbar_init(&w_full[s], 1); mbar_init(&w_empty[s], 1); }
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) { tmem_alloc(tmem_slot, G::TMEM_COLS); tmem_relinquish(); }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_pairs = (p.n_tiles + 1) >> 1;

  if (warp == 1) {
    // ------------------------------------------------ weight producer
    if (lane == 0) {
      if (resident) {
        uint32_t total = 0;
        for (int j = 0; j < p.n_jobs; ++j) total += G::MAT_BYTES;
        mbar_arrive_expect_tx(&w_full[0], total);
        for (int j = 0; j < p.n_jobs; ++j)
          bulk_g2s(ring + j * G::MAT_BYTES, p.wmats + (size_t)p.job_mat[j] * p.mat_bytes, G::MAT_BYTES, &w_full[0]);
      } else {
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
      }
    }
    __syncwarp();
  } else if (warp == 0) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t a_use[2] = {0, 0};
      uint32_t seq = 0;
      bool ok = true;
      if (resident) ok = bounded_wait(&w_full[0], 0, abort_flag, p.err);
      for (int pair = blockIdx.x; ok && pair < n_pairs; pair += gridDim.x) {
        const bool has1 = (2 * pair + 1) < p.n_tiles;
        for (int j = 0; j < p.n_jobs && ok; ++j, ++seq) {
          const int st = resident ? j : (int)(seq % G::STAGES);
          if (!resident) ok = bounded_wait(&w_full[st], (seq / G::STAGES) & 1, abort_flag, p.err);
          if (!ok) break;
          const uint32_t wb = smem_u32(ring + st * G::MAT_BYTES);
          for (int s = 0; s < 2 && ok; ++s) {
            if (s == 1 && !has1) break;
            ok = bounded_wait(&a_full[s], a_use[s] & 1, abort_flag, p.err);
            a_use[s]++;
            if (!ok) break;
            tc_fence_after();
            const uint32_t d = tmem_base + s * G::SLOT_COLS;
            const uint32_t ahi = d + H, alo = d + H + H / 2;
#pragma unroll
            for (int ks = 0; ks < H / 16; ++ks) {
              const uint32_t off = (ks >> 2) * (H * 128) + (ks & 3) * 32;
              const uint64_t bh = sdesc_kmajor_sw128(wb + off);
              const uint64_t bl = sdesc_kmajor_sw128(wb + G::PART_BYTES + off);
              const uint32_t acc = (p.job_acc[j] || ks > 0) ? 1u : 0u;
              mma_bf16_ts(d, ahi + ks * 8, bh, G::IDESC, acc);
              mma_bf16_ts(d, ahi + ks * 8, bl, G::IDESC, 1u);
              mma_bf16_ts(d, alo + ks * 8, bh, G::IDESC, 1u);
            }
            mma_commit(&d_full[s]);
          }
          if (!resident && ok) mma_commit(&w_empty[st]);
        }
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ row workers
    const int wi = warp - 2;                 // 0..15
    const int slot = wi >> 3;
    const int half = (wi >> 2) & 1;
    const int quarter = warp & 3;            // TMEM lane quarter of this warp
    const int trow = quarter * 32 + lane;    // row inside the tile
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t d_addr = tmem_base + slot * G::SLOT_COLS + lane_off + half * HH;
    const uint32_t ahi_addr = tmem_base + slot * G::SLOT_COLS + H + lane_off + half * (HH / 2);
    const uint32_t alo_addr = ahi_addr + H / 2;
    float* red_slot = red + slot * (2 * 2 * 128);
    uint32_t d_use = 0, xbuf = 0;
    const int c0 = half * HH;                // first column of this thread

    auto arrive_a = [&]() {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&a_full[slot]);
    };
    auto wait_d = [&]() -> bool {
      const bool ok = bounded_wait(&d_full[slot], d_use & 1, abort_flag, p.err);   // never early-exits a tile
      d_use++;
      tc_fence_after();
      return ok;
    };
    auto load_d_add = [&](float* v) {        // v += D (this thread's HH columns)
#pragma unroll
      for (int c = 0; c < HH; c += 16) {
        float t[16];
        tmem_ld16(d_addr + c, t);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 16; ++i) v[c + i] += t[i];
      }
    };
    auto store_a = [&](const float* v) {     // split to bf16 hi/lo, write A operand
#pragma unroll
      for (int c = 0; c < HH; c += 16) {
        uint32_t hi[8], lo[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) split_bf16x2(v[c + 2 * i], v[c + 2 * i + 1], hi[i], lo[i]);
        tmem_st8(ahi_addr + c / 2, hi);
        tmem_st8(alo_addr + c / 2, lo);
      }
      tmem_st_wait();
    };
    auto xchg = [&](float mine) -> float {   // value of the other column half of this row
      float* b = red_slot + xbuf * 256;
      b[half * 128 + trow] = mine;
      named_bar_sync(1 + slot, 256);
      const float other = b[(1 - half) * 128 + trow];
      xbuf ^= 1;
      return other;
    };
    auto ln_relu = [&](float* v, const float* gamma, const float* beta) {
      float s = 0.f;
#pragma unroll
      for (int i = 0; i < HH; ++i) s += v[i];
      s += xchg(s);
      const float mean = s * (1.0f / H);
      float q = 0.f;
#pragma unroll
      for (int i = 0; i < HH; ++i) { const float dd = v[i] - mean; q += dd * dd; }
      q += xchg(q);
      const float rstd = rsqrtf(q * (1.0f / H) + p.eps);
#pragma unroll
      for (int i = 0; i < HH; ++i) v[i] = fmaxf(fmaf((v[i] - mean) * rstd, gamma[c0 + i], beta[c0 + i]), 0.f);
    };
    auto add_vec = [&](float* v, const float* b) {
#pragma unroll
      for (int i = 0; i < HH; ++i) v[i] += b[c0 + i];
    };
    auto load_row = [&](float* v, const float* base, bool ok) {   // v = base[c0 .. c0+HH)
      if (ok) {
        const float4* s4 = reinterpret_cast<const float4*>(base + c0);
#pragma unroll
        for (int i = 0; i < HH / 4; ++i) { const float4 t = s4[i]; v[4*i] = t.x; v[4*i+1] = t.y; v[4*i+2] = t.z; v[4*i+3] = t.w; }
      } else {
#pragma unroll
        for (int i = 0; i < HH; ++i) v[i] = 0.f;
      }
    };
    auto add_row = [&](float* v, const float* base) {
      const float4* s4 = reinterpret_cast<const float4*>(base + c0);
#pragma unroll
      for (int i = 0; i < HH / 4; ++i) { const float4 t = s4[i]; v[4*i] += t.x; v[4*i+1] += t.y; v[4*i+2] += t.z; v[4*i+3] += t.w; }
    };
    auto store_row = [&](float* base, const float* v) {
      float4* d4 = reinterpret_cast<float4*>(base + c0);
#pragma unroll
      for (int i = 0; i < HH / 4; ++i) d4[i] = make_float4(v[4*i], v[4*i+1], v[4*i+2], v[4*i+3]);
    };
    // First layer of an encoder on CUDA cores: v = W1 f + b1, W1 [H, nf] row-major in smem.
    auto small_linear = [&](float* v, const float* f, int nf, const float* W1, const float* b1) {
#pragma unroll
      for (int i = 0; i < HH; ++i) {
        float acc = b1[c0 + i];
        for (int k = 0; k < nf; ++k) acc = fmaf(W1[(c0 + i) * nf + k], f[k], acc);
        v[i] = acc;
      }
    };

    const int L = p.n_layers;
    bool ok = true;
    for (int pair = blockIdx.x; ok && pair < n_pairs; pair += gridDim.x) {
      const int tile = 2 * pair + slot;
      if (tile >= p.n_tiles) break;
      const int row = tile * kTileRows + trow;
      const bool valid = row < p.n_rows;
      float v[HH];

      if constexpr (KIND == TileKind::EdgeUpdate || KIND == TileKind::Classifier) {
        // vec layout: [gamma1, beta1, (b_l, gamma_l, beta_l) for l = 2..L, (w_o, b_o)]
        load_row(v, p.e + (size_t)row * H, valid);
        store_a(v); arrive_a();
        // layer-1 pre-activation terms of the endpoints (P_d carries b1)
        if (valid) {
          const int s = p.src_sorted[row], d = p.dst_sorted[row];
          load_row(v, p.ps + (size_t)s * H, true);
          add_row(v, p.pd + (size_t)d * H);
        } else {
#pragma unroll
          for (int i = 0; i < HH; ++i) v[i] = 0.f;
        }
        for (int l = 1; l <= L; ++l) {
          if (l > 1) {
#pragma unroll
            for (int i = 0; i < HH; ++i) v[i] = 0.f;
          }
          ok &= wait_d();
          load_d_add(v);
          const float* vb = vecs + (l == 1 ? 0 : (2 + 3 * (l - 2)) * H);
          if (l > 1) { add_vec(v, vb); vb += H; }
          ln_relu(v, vb, vb + H);
          if (l < L) { store_a(v); arrive_a(); }
        }
        if constexpr (KIND == TileKind::EdgeUpdate) {
          if (ok && valid) store_row(p.e + (size_t)row * H, v);
        } else {
          const float* wo = vecs + (2 + 3 * (L - 1)) * H;
          float z = 0.f;
#pragma unroll
          for (int i = 0; i < HH; ++i) z = fmaf(v[i], wo[c0 + i], z);
          z += xchg(z);
          if (ok && valid && half == 0) {
            const float logit = z + wo[H];
            const float sc = 1.0f / (1.0f + __expf(-logit));
            const bool good = p.key_sorted[row] < p.n_nodes;
            p.scores[p.perm[row]] = good ? sc : __int_as_float(0x7fc00000);
          }
        }
      } else if constexpr (KIND == TileKind::EdgeEncoder) {
        // vec layout: [W1 (H x 2), b1, gamma1, beta1, (b_l, gamma_l, beta_l) for l = 2..L]
        float f[2] = {0.f, 0.f};
        if (valid) {
          const int s = p.src_sorted[row], d = p.dst_sorted[row];
          const float* xs = p.x + (size_t)s * p.x_stride;
          const float* xd = p.x + (size_t)d * p.x_stride;
          f[0] = xd[0] - xs[0];
          float dphi = xd[1] - xs[1];
          if (dphi > 1.0f) dphi -= 2.0f;
          if (dphi <= -1.0f) dphi += 2.0f;
          f[1] = dphi;
        }
        const float* W1 = vecs;
        const float* vb = vecs + 2 * H;
        small_linear(v, f, 2, W1, vb);
        ln_relu(v, vb + H, vb + 2 * H);
        store_a(v); arrive_a();
        for (int l = 2; l <= L; ++l) {
#pragma unroll
          for (int i = 0; i < HH; ++i) v[i] = 0.f;
          ok &= wait_d();
          load_d_add(v);
          const float* vl = vb + 3 * (l - 1) * H;
          add_vec(v, vl);
          ln_relu(v, vl + H, vl + 2 * H);
          if (l < L) { store_a(v); arrive_a(); }
        }
        if (ok && valid) store_row(p.e + (size_t)row * H, v);
      } else {
        // NodeEncoder / NodeUpdate.
        // vec layout: [W1 (H x n_feat) if encoder], (b_l, gamma_l, beta_l) for l = 1..L, b1_edge
        const float* vb = vecs + (KIND == TileKind::NodeEncoder ? p.n_feat * H : 0);
        int l0;
        if constexpr (KIND == TileKind::NodeEncoder) {
          float f[16];
          for (int k = 0; k < 16; ++k) f[k] = (valid && k < p.n_feat) ? p.x[(size_t)row * p.x_stride + k] : 0.f;
          small_linear(v, f, p.n_feat, vecs, vb);
          ln_relu(v, vb + H, vb + 2 * H);
          store_a(v); arrive_a();
          l0 = 2;
        } else {
          load_row(v, p.h + (size_t)row * H, valid);
          store_a(v); arrive_a();                       // job: D = h * W_nh^T
#pragma unroll
          for (int i = 0; i < HH; ++i) v[i] = 0.f;
          if (valid) {                                  // a_j: CSR segment sum, fixed order
            const int k0 = p.rowptr[row], k1 = p.rowptr[row + 1];
            for (int k = k0; k < k1; ++k) add_row(v, p.e + (size_t)k * H);
          }
          ok &= wait_d();                // A free again
          store_a(v); arrive_a();                       // job: D += a * W_na^T
          l0 = 1;
        }
        for (int l = l0; l <= L; ++l) {
#pragma unroll
          for (int i = 0; i < HH; ++i) v[i] = 0.f;
          ok &= wait_d();
          load_d_add(v);
          const float* vl = vb + 3 * (l - 1) * H;
          add_vec(v, vl);
          ln_relu(v, vl + H, vl + 2 * H);
          store_a(v); arrive_a();                       // next layer, or the P_s job
        }
        if (ok && valid) store_row(p.h + (size_t)row * H, v);
        // P_s = W_s h (no bias)
#pragma unroll
        for (int i = 0; i < HH; ++i) v[i] = 0.f;
        ok &= wait_d();
        load_d_add(v);
        if (ok && valid) store_row(p.ps + (size_t)row * H, v);
        arrive_a();                                     // D read; A (= h) unchanged -> P_d job
        // P_d = W_d h + b1 (edge-side bias)
#pragma unroll
        for (int i = 0; i < HH; ++i) v[i] = 0.f;
        ok &= wait_d();
        load_d_add(v);
        add_vec(v, vb + 3 * L * H);
        if (ok && valid) store_row(p.pd + (size_t)row * H, v);
      }
      if (!ok) break;                        // leave only between tiles
    }
    __syncwarp();
  }

  // teardown: every role reaches this point (waits are bounded)
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, G::TMEM_COLS);
  }
}

}  // namespace gnn
