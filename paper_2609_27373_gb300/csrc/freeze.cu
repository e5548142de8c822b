// Freeze-A control with a stored distribution (appendix "Experimental
// details", intervention controls): the support W of WISE with the
// within-support attention of a past step t0 frozen,
//   Abar_ij = A(t0)_ij [b(j) in W_q(i)] / sum_k A(t0)_ik [b(k) in W_q(i)],
//   O(t) = Abar V(t).
// Abar is the softmax over the support of step t0's logits, so
// freeze_probs_kernel computes it once from Q(t0) and K(t0) and stores it as
// Abar = diag(inv_l) P: P = 2^(s - m) relative to each row's maximum (so the
// largest term of a row is exactly 1) as bf16 128 x 128 tiles in the order of
// the support walk, and inv_l = 1 / (row sum) in fp32 per row.
// frozen_pv_kernel then runs each late step as a block-sparse P V product (no
// logits, no softmax), streaming the stored tiles from HBM, and scales each
// row of O by inv_l.
//
// Both kernels walk a unit's key tiles (a unit is a 128-row query tile of one
// (batch, head)) with the attention kernel's iterator, so tile t of a unit is
// the same key tile in both; in P the units follow the (batch, head, query
// tile) order.  Warps 0-3 own the 128 rows (TMEM lanes).  The probabilities
// kernel takes one unit per CTA and lane 0 of warp 4 issues its TMA loads and
// tcgen05 MMAs; the P V kernel is persistent (described there).
#include "attn_kernel.cuh"

namespace wise {
namespace {

template <int D>
struct FzCfg {
  static constexpr int kBoxes = (D + 63) / 64;
  static constexpr int kQBytes = kBoxes * 128 * 128;   // one 128-row Q tile
  static constexpr int kKBytes = kBoxes * 128 * 128;   // one 128-key K or V tile
  static constexpr int kPBytes = 2 * 128 * 128;        // one 128 x 128 bf16 P tile (two 64-column boxes)
  static constexpr int kThreads = 160;
  static constexpr int kRing = 3;
  static constexpr int kSmemProbs = kQBytes + kRing * kKBytes + 1024;
  static constexpr int kSmemPV = kRing * (kPBytes + kKBytes) + 1024;
  static constexpr int kIssuerWarp = 4;
};

template <int BLK>
__device__ __forceinline__ int walk_length(const AttnParams& p, int b, int kvh, int qt) {
  auto it = make_iter<BLK, kSparse>(p, b, kvh, qt);
  int kt, n = 0;
  uint32_t mask;
  while (it.next(kt, mask)) ++n;
  return n;
}

struct FzShared {
  uint64_t q_full, full[3], empty[3], s_full[2], s_free[2], done;
  uint32_t tmem_base;
  int abort;
  int n_tiles;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// ---------------------------------------------------------------- probabilities
// Two passes over the unit's key tiles: the first forms each row's maximum m
// and sum l over the support (online), the second recomputes S and stores
// P = 2^(s * scale_log2 - m) (0 where masked) and inv_l = 1 / l (0 for rows
// with no admissible key).
template <int D, int BLK>
__global__ void __launch_bounds__(160, 1)
    freeze_probs_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                        const AttnParams p, __nv_bfloat16* P, float* inv_l, int tile_cap) {
  using C = FzCfg<D>;
  constexpr int S = kTileN / BLK;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* q_stage = align1024(smem_raw);
  uint8_t* ring = q_stage + C::kQBytes;
  __shared__ FzShared sh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int u = blockIdx.x;
  int b, h, qt;
  decode_unit(p, u, b, h, qt);
  const int kvh = h / p.group;
  if (threadIdx.x == 0) {
    sh.abort = 0;
    mbar_init(&sh.q_full, 1);
    for (int i = 0; i < 3; ++i) {
      mbar_init(&sh.full[i], 1);
      mbar_init(&sh.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.s_full[i], 1);
      mbar_init(&sh.s_free[i], 4);
    }
    mbar_init(&sh.done, 1);
    sh.n_tiles = walk_length<BLK>(p, b, kvh, qt);
    fence_mbar_init();
  }
  if (warp == C::kIssuerWarp) {
    tmem_alloc(&sh.tmem_base, 256);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  const int n = sh.n_tiles;
  volatile int* abort = &sh.abort;

  if (warp == C::kIssuerWarp) {
    if (lane == 0 && n > 0) {
      const int z = b * p.n_kv_heads + kvh;
      const int total = 2 * n;
      bool ok = true;
      mbar_arrive_expect_tx(&sh.q_full, C::kQBytes);
      for (int i = 0; i < C::kBoxes; ++i)
        tma_load_3d(q_stage + i * 128 * 128, &mapQ, &sh.q_full, 64 * i, qt * 128, b * p.n_heads + h);
      // K loads run up to two tiles ahead of the products; the walk restarts
      // for the second pass.
      auto it = make_iter<BLK, kSparse>(p, b, kvh, qt);
      int jl = 0;
      auto load_next = [&]() -> bool {
        int kt;
        uint32_t mask;
        if (jl == n) it = make_iter<BLK, kSparse>(p, b, kvh, qt);
        if (!it.next(kt, mask)) return false;  // cannot happen: the walk has n tiles
        const int slot = jl % 3;
        if (jl >= 3 && !mbar_wait(&sh.empty[slot], ((jl / 3) - 1) & 1, abort)) return false;
        mbar_arrive_expect_tx(&sh.full[slot], C::kKBytes);
        for (int i = 0; i < C::kBoxes; ++i)
          tma_load_3d(ring + slot * C::kKBytes + i * kTileN * 128, &mapK, &sh.full[slot], 64 * i, kt * kTileN, z);
        ++jl;
        return true;
      };
      for (int i = 0; i < 2 && i < total && ok; ++i) ok = load_next();
      constexpr uint32_t idesc = idesc_bf16_f32(128, kTileN, false, false);
      const uint64_t a0 = smem_desc_sw128(smem_u32(q_stage), 16, 1024);
      if (ok && !mbar_wait(&sh.q_full, 0, abort)) ok = false;
      for (int j = 0; j < total && ok; ++j) {
        if (jl < total && jl <= j + 2 && !load_next()) {
          ok = false;
          break;
        }
        const int slot = j % 3;
        if (!mbar_wait(&sh.full[slot], (j / 3) & 1, abort)) {
          ok = false;
          break;
        }
        // S buffer j & 1 was read by the rows at tile j - 2.
        if (j >= 2 && !mbar_wait(&sh.s_free[j & 1], ((j - 2) >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint64_t b0 = smem_desc_sw128(smem_u32(ring + slot * C::kKBytes), 16, 1024);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t a_off = ((kk >> 2) * (128 * 128) + (kk & 3) * 32) >> 4;
          const uint32_t b_off = ((kk >> 2) * (kTileN * 128) + (kk & 3) * 32) >> 4;
          umma_bf16_ss(tmem + (j & 1) * 128, a0 + a_off, b0 + b_off, idesc, kk > 0 ? 1u : 0u);
        }
        umma_commit(&sh.s_full[j & 1]);
        umma_commit(&sh.empty[slot]);
      }
      if (!ok) raise_status(p, &sh.abort, kStatusTimeout);
      umma_commit(&sh.done);
      int never = 0;
      mbar_wait(&sh.done, 0, &never);
      // Copies already issued land before shared memory is released.
      for (int t = max(0, jl - 3); t < jl; ++t) mbar_wait(&sh.full[t % 3], (t / 3) & 1, &never);
      mbar_wait(&sh.q_full, 0, &never);
    }
  } else {
    const int r = threadIdx.x;  // row of the tile = TMEM lane
    const int wq = r >> 5;
    const uint32_t lane_tmem = tmem + ((uint32_t)(wq * 32) << 16);
    const int row = qt * 128 + r;
    const int qsub = r / BLK;
    float m = -INFINITY, l = 0.0f;
    int j = 0;
    bool ok = true;
    for (int pass = 0; pass < 2 && ok; ++pass) {
      auto it = make_iter<BLK, kSparse>(p, b, kvh, qt);
      int kt, t = 0;
      uint32_t mask;
      while (it.next(kt, mask)) {
        if (!warp_wait(&sh.s_full[j & 1], (j >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t sub = (mask >> (qsub * S)) & ((1u << S) - 1u);
        float s[kTileN];
        load_s_row<BLK>(lane_tmem + (j & 1) * 128, s, sub, row - kt * kTileN);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.s_free[j & 1]);
        if (pass == 0) {
          const float mt = row_max(s) * p.scale_log2;
          const float mn = fmaxf(m, mt);
          if (mn != -INFINITY) {
            l = (m == -INFINITY ? 0.0f : l * ex2_approx(m - mn)) + exp2_scaled(s, p.scale_log2, mn);
            m = mn;
          }
        } else if (t < tile_cap) {
          const size_t tile = ((size_t)(b * p.n_heads + h) * p.n_qtiles + qt) * tile_cap + t;
          uint4* dst = reinterpret_cast<uint4*>(P + (tile * 128 + r) * 128);
          if (m == -INFINITY) {
#pragma unroll
            for (int c = 0; c < kTileN / 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
          } else {
            exp2_scaled(s, p.scale_log2, m);
#pragma unroll
            for (int c = 0; c < kTileN / 8; ++c)
              dst[c] = make_uint4(pack_bf16x2(s[8 * c], s[8 * c + 1]), pack_bf16x2(s[8 * c + 2], s[8 * c + 3]),
                                  pack_bf16x2(s[8 * c + 4], s[8 * c + 5]), pack_bf16x2(s[8 * c + 6], s[8 * c + 7]));
          }
        }
        ++j;
        ++t;
      }
      if (pass == 0) {
        const size_t unit = (size_t)(b * p.n_heads + h) * p.n_qtiles + qt;
        inv_l[unit * 128 + r] = l > 0.0f ? 1.0f / l : 0.0f;
      }
    }
    if (!ok) raise_status(p, &sh.abort, kStatusTimeout);
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == C::kIssuerWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, 256);
  }
}

// ------------------------------------------------------------- frozen P V
// Persistent: CTA c takes the units k * G + c (even rounds k) and
// k * G + G - 1 - c (odd rounds), longest causal prefix first.  Warp 4
// streams the P and V tiles of all its units through a three-stage ring, warp
// 5 issues O += P_t V_t into one of two TMEM accumulators (alternating per
// unit with tiles), and warps 0-3 read each finished accumulator, scale its
// rows by inv_l and store them while the next unit accumulates.
struct PvShared {
  uint64_t full[3], empty[3], o_full[2], o_free[2], done;
  uint32_t tmem_base;
  int abort;
};

template <int D, int BLK>
__global__ void __launch_bounds__(192, 1)
    frozen_pv_kernel(const __grid_constant__ CUtensorMap mapP, const __grid_constant__ CUtensorMap mapV,
                     const AttnParams p, const float* inv_l, int tile_cap) {
  using C = FzCfg<D>;
  constexpr int kStage = C::kPBytes + C::kKBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = align1024(smem_raw);
  __shared__ PvShared sh;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = gridDim.x, c = blockIdx.x;
  auto unit_of = [&](int k) { return k * G + ((k & 1) ? G - 1 - c : c); };
  if (threadIdx.x == 0) {
    sh.abort = 0;
    for (int i = 0; i < 3; ++i) {
      mbar_init(&sh.full[i], 1);
      mbar_init(&sh.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.o_full[i], 1);
      mbar_init(&sh.o_free[i], 4);
    }
    mbar_init(&sh.done, 1);
    fence_mbar_init();
  }
  if (warp == 5) {
    tmem_alloc(&sh.tmem_base, 256);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sh.tmem_base;
  volatile int* abort = &sh.abort;

  if (warp == 4) {
    if (lane == 0) {
      int jl = 0;
      bool ok = true;
      for (int k = 0; ok && k * G < p.n_units; ++k) {
        const int u = unit_of(k);
        if (u >= p.n_units) continue;
        int b, h, qt;
        decode_unit(p, u, b, h, qt);
        const int kvh = h / p.group;
        const int z = b * p.n_kv_heads + kvh;
        const int p_base = ((b * p.n_heads + h) * p.n_qtiles + qt) * tile_cap;
        auto it = make_iter<BLK, kSparse>(p, b, kvh, qt);
        int kt;
        uint32_t mask;
        for (int t = 0; t < tile_cap && it.next(kt, mask); ++t) {
          const int slot = jl % 3;
          if (jl >= 3 && !mbar_wait(&sh.empty[slot], ((jl / 3) - 1) & 1, abort)) {
            ok = false;
            break;
          }
          uint8_t* st = ring + slot * kStage;
          mbar_arrive_expect_tx(&sh.full[slot], kStage);
          for (int i = 0; i < 2; ++i) tma_load_3d(st + i * 128 * 128, &mapP, &sh.full[slot], 64 * i, 0, p_base + t);
          for (int i = 0; i < C::kBoxes; ++i)
            tma_load_3d(st + C::kPBytes + i * kTileN * 128, &mapV, &sh.full[slot], 64 * i, kt * kTileN, z);
          ++jl;
        }
      }
      if (!ok) {
        raise_status(p, &sh.abort, kStatusTimeout);
        int never = 0;
        for (int t = max(0, jl - 3); t < jl; ++t) mbar_wait(&sh.full[t % 3], (t / 3) & 1, &never);
      }
    }
  } else if (warp == 5) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, D, false, true);
      int j = 0, ni = 0;
      bool ok = true;
      for (int k = 0; ok && k * G < p.n_units; ++k) {
        const int u = unit_of(k);
        if (u >= p.n_units) continue;
        int b, h, qt;
        decode_unit(p, u, b, h, qt);
        const int n = min(walk_length<BLK>(p, b, h / p.group, qt), tile_cap);
        if (n == 0) continue;
        const int ob = ni & 1;
        // Accumulator ob was last read by the epilogue of unit ni - 2.
        if (ni >= 2 && !mbar_wait(&sh.o_free[ob], ((ni - 2) >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        for (int t = 0; t < n; ++t, ++j) {
          const int slot = j % 3;
          if (!mbar_wait(&sh.full[slot], (j / 3) & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint32_t st = smem_u32(ring + slot * kStage);
          const uint64_t a0 = smem_desc_sw128(st, 16, 1024);
          const uint64_t b0 = smem_desc_sw128(st + C::kPBytes, kTileN * 128, 1024);
#pragma unroll
          for (int kk = 0; kk < kTileN / 16; ++kk) {
            const uint32_t a_off = ((kk >> 2) * (128 * 128) + (kk & 3) * 32) >> 4;
            umma_bf16_ss(tmem + ob * 128, a0 + a_off, b0 + ((kk * 2048) >> 4), idesc, (t > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(&sh.empty[slot]);
        }
        if (!ok) break;
        umma_commit(&sh.o_full[ob]);
        ++ni;
      }
      if (!ok) raise_status(p, &sh.abort, kStatusTimeout);
      umma_commit(&sh.done);
      int never = 0;
      mbar_wait(&sh.done, 0, &never);
    }
  } else {
    const int r = threadIdx.x;  // row of the tile = TMEM lane
    const int wq = r >> 5;
    const uint32_t lane_tmem = tmem + ((uint32_t)(wq * 32) << 16);
    int ni = 0;
    bool ok = true;
    for (int k = 0; ok && k * G < p.n_units; ++k) {
      const int u = unit_of(k);
      if (u >= p.n_units) continue;
      int b, h, qt;
      decode_unit(p, u, b, h, qt);
      const int n = min(walk_length<BLK>(p, b, h / p.group, qt), tile_cap);
      const int row = qt * 128 + r;
      float o[D];
      if (n > 0) {
        const int ob = ni & 1;
        if (!warp_wait(&sh.o_full[ob], (ni >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        tmem_load_row<D>(lane_tmem + ob * 128, o);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh.o_free[ob]);
        ++ni;
      }
      if (row < p.seqlen) {
        const float f = inv_l[((size_t)(b * p.n_heads + h) * p.n_qtiles + qt) * 128 + r];
        uint4* dst = reinterpret_cast<uint4*>(p.O + ((size_t)(b * p.n_heads + h) * p.seqlen + row) * D);
#pragma unroll
        for (int c8 = 0; c8 < D / 8; ++c8)
          dst[c8] = n > 0 ? make_uint4(pack_bf16x2(o[8 * c8] * f, o[8 * c8 + 1] * f),
                                       pack_bf16x2(o[8 * c8 + 2] * f, o[8 * c8 + 3] * f),
                                       pack_bf16x2(o[8 * c8 + 4] * f, o[8 * c8 + 5] * f),
                                       pack_bf16x2(o[8 * c8 + 6] * f, o[8 * c8 + 7] * f))
                          : make_uint4(0u, 0u, 0u, 0u);
      }
    }
    if (!ok) raise_status(p, &sh.abort, kStatusTimeout);
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, 256);
  }
}

template <int D, int BLK>
cudaError_t launch_probs_instance(const FreezeLaunch& L) {
  auto kern = freeze_probs_kernel<D, BLK>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, FzCfg<D>::kSmemProbs);
  if (e != cudaSuccess) return e;
  kern<<<L.p.n_units, FzCfg<D>::kThreads, FzCfg<D>::kSmemProbs, L.stream>>>(L.mapQ, L.mapK, L.p, L.P, L.inv_l,
                                                                             L.tile_cap);
  return cudaGetLastError();
}

template <int D, int BLK>
cudaError_t launch_pv_instance(const FreezeLaunch& L) {
  auto kern = frozen_pv_kernel<D, BLK>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, FzCfg<D>::kSmemPV);
  if (e != cudaSuccess) return e;
  kern<<<L.grid, 192, FzCfg<D>::kSmemPV, L.stream>>>(L.mapP, L.mapV, L.p, L.inv_l, L.tile_cap);
  return cudaGetLastError();
}

template <int D>
cudaError_t probs_for_dim(int block, const FreezeLaunch& L) {
  return block == 128 ? launch_probs_instance<D, 128>(L)
                      : block == 64 ? launch_probs_instance<D, 64>(L) : launch_probs_instance<D, 32>(L);
}

template <int D>
cudaError_t pv_for_dim(int block, const FreezeLaunch& L) {
  return block == 128 ? launch_pv_instance<D, 128>(L)
                      : block == 64 ? launch_pv_instance<D, 64>(L) : launch_pv_instance<D, 32>(L);
}

}  // namespace

cudaError_t launch_freeze_probs(int head_dim, int block, const FreezeLaunch& L) {
  switch (head_dim) {
    case 64: return probs_for_dim<64>(block, L);
    case 96: return probs_for_dim<96>(block, L);
    default: return probs_for_dim<128>(block, L);
  }
}

cudaError_t launch_frozen_pv(int head_dim, int block, const FreezeLaunch& L) {
  switch (head_dim) {
    case 64: return pv_for_dim<64>(block, L);
    case 96: return pv_for_dim<96>(block, L);
    default: return pv_for_dim<128>(block, L);
  }
}

}  // namespace wise
