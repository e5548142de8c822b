// Causal flash attention on tcgen05 tensor cores, in three variants:
//   kDense      O = softmax(Q K^T * scale + M) V                  (Eq. 2)
//   kDenseMass  the same, plus the block attention mass of the step (Eq. 5)
//               accumulated into blockmass
//   kSparse     key blocks restricted to the selected support      (Eqs. 7-8)
//
// Work decomposition.  A unit is one 128-row query tile of one (batch, head).
// The grid is persistent (one CTA per SM); CTA c takes units c, c + grid, ...
// in order of decreasing causal length.  Each unit walks its list of key
// tiles (BN = block keys each): every tile of the causal prefix (dense), or
// the blocks of the support (sparse; with block 64 a query tile covers two
// query blocks and walks the union of their lists, masking per half).
//
// Warp roles (192 threads):
//   warps 0-3  softmax: thread t owns query row t of the tile (= TMEM lane t).
//              It reads its row of S from TMEM, keeps the running max and sum
//              (online softmax in the log2 domain, with the rescale of O
//              skipped unless the max grows by more than 2^8), writes P as
//              bf16 into shared memory, and runs the epilogue: O / l to
//              global memory, and for kDenseMass the block masses.
//   warp 4     TMA producer: Q tile (double-buffered across units) and K/V
//              tiles (kStages-deep ring).
//   warp 5     MMA issuer: S = Q K^T into one of two TMEM S buffers, then
//              O += P V into the TMEM O accumulator, one tile behind, so the
//              tensor core computes S(j+1) while the softmax works on S(j).
//
// Block mass (Eq. 5) needs each row's final normaliser, which is known only
// after the last tile.  For every tile the softmax thread stores
// lc = m + log2(sum_{j in tile} 2^(s_j - m)) (its row's partial mass in log2
// units, m the running max at the time) in a per-CTA scratch row; the
// epilogue turns it into A-mass 2^(lc - lse), sums the 128 (or 2 x 64) rows
// of each query block with warp shuffles and a fixed-order cross-warp sum
// (deterministic), divides by B and writes or accumulates blockmass.
#pragma once

#include <cuda_bf16.h>
#include <limits.h>
#include <stdint.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace wise {

template <int D, int BN>
struct AttnCfg {
  static constexpr int kBoxes = (D + 63) / 64;          // 64-column TMA boxes per row tile
  static constexpr int kQBytes = kBoxes * 128 * 128;    // one 128-row Q tile
  static constexpr int kKVBytes = kBoxes * BN * 128;    // one BN-row K or V tile
  static constexpr int kPBytes = (BN / 64) * 128 * 128; // P tile, 128 x BN bf16
  static constexpr int kStages = (D <= 64) ? 4 : 2;
  static constexpr int kSmemBytes = 2 * kQBytes + 2 * kStages * kKVBytes + kPBytes + 1024;
  // At least 116 KB so that a single CTA resides per SM (it owns all 512
  // TMEM columns).
  static constexpr int kSmemLaunch = kSmemBytes > 116 * 1024 ? kSmemBytes : 116 * 1024;
  static constexpr uint32_t kTmemO = 2 * BN;            // S buffers at columns 0 and BN
  static constexpr uint32_t kTmemCols = 512;
  static constexpr int kThreads = 192;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
  static_assert(2 * BN + D <= 512, "TMEM budget");
};

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Key tiles of one unit in ascending order.  Dense: 0..last.  Sparse: the
// support list of the unit's query block (block 128), or the merge of the
// lists of its two query blocks (block 64); `bits` says which half of the
// 128 query rows may attend the tile.  Entries that are negative, beyond the
// query block, or not strictly ascending are skipped and flagged in `bad`.
struct TileIter {
  int dense, cur, last;
  const int32_t* la;
  const int32_t* lb;
  int na, ia, lima, preva, pend_a;
  int nb, ib, limb, prevb, pend_b;
  int bad;

  __device__ __forceinline__ int pull(const int32_t* l, int n, int& i, int lim, int& prev) {
    while (i < n) {
      const int v = __ldg(l + i);
      ++i;
      if (v >= 0 && v <= lim && v > prev) {
        prev = v;
        return v;
      }
      bad = 1;
    }
    return INT_MAX;
  }

  __device__ __forceinline__ bool next(int& kb, int& bits) {
    if (dense) {
      if (cur > last) return false;
      kb = cur++;
      bits = 3;
      return true;
    }
    if (pend_a == INT_MAX && pend_b == INT_MAX) return false;
    if (pend_a < pend_b) {
      kb = pend_a;
      bits = 1;
      pend_a = pull(la, na, ia, lima, preva);
    } else if (pend_b < pend_a) {
      kb = pend_b;
      bits = 2;
      pend_b = pull(lb, nb, ib, limb, prevb);
    } else {
      kb = pend_a;
      bits = 3;
      pend_a = pull(la, na, ia, lima, preva);
      pend_b = pull(lb, nb, ib, limb, prevb);
    }
    return true;
  }
};

__device__ __forceinline__ int clamp_count(int n, int cap, int& bad) {
  if (n < 0 || n > cap) {
    bad = 1;
    return n < 0 ? 0 : cap;
  }
  return n;
}

template <int BN, int MODE>
__device__ __forceinline__ TileIter make_iter(const AttnParams& p, int b, int kvh, int qt) {
  TileIter it;
  it.bad = 0;
  if (MODE != kSparse) {
    it.dense = 1;
    it.cur = 0;
    const int last_row = min(qt * 128 + 127, p.seqlen - 1);
    it.last = last_row / BN;
    it.pend_a = it.pend_b = INT_MAX;
    return it;
  }
  it.dense = 0;
  constexpr int kQbPerTile = 128 / BN;
  const int q0 = qt * kQbPerTile;
  const size_t row0 = ((size_t)b * p.n_kv_heads + kvh) * p.n_blocks + q0;
  it.la = p.idx + row0 * p.cap;
  it.na = clamp_count(__ldg(p.counts + row0), p.cap, it.bad);
  it.ia = 0;
  it.lima = q0;
  it.preva = -1;
  if (kQbPerTile == 2 && q0 + 1 < p.n_blocks) {
    it.lb = p.idx + (row0 + 1) * p.cap;
    it.nb = clamp_count(__ldg(p.counts + row0 + 1), p.cap, it.bad);
  } else {
    it.lb = it.la;
    it.nb = 0;
  }
  it.ib = 0;
  it.limb = q0 + 1;
  it.prevb = -1;
  it.pend_a = it.pull(it.la, it.na, it.ia, it.lima, it.preva);
  it.pend_b = it.pull(it.lb, it.nb, it.ib, it.limb, it.prevb);
  return it;
}

__device__ __forceinline__ void decode_unit(const AttnParams& p, int u, int& b, int& h, int& qt) {
  const int bh_count = p.batch * p.n_heads;
  qt = p.n_qtiles - 1 - u / bh_count;  // longest causal prefix first
  const int bh = u % bh_count;
  b = bh / p.n_heads;
  h = bh % p.n_heads;
}

struct SharedBarriers {
  uint64_t q_full[2], q_empty[2];
  uint64_t k_full[4], v_full[4], kv_empty[4];
  uint64_t s_full[2];
  uint64_t p_full, o_full, mma_done;
  uint64_t epi;  // the four softmax warps meet here in the block-mass epilogue
  uint32_t tmem_base;
  int abort;
};

// mbar_wait whose outcome is the same for every lane of the warp (all lanes
// must call it together): a lane that gave up makes the whole warp give up.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

__device__ __forceinline__ void raise_status(const AttnParams& p, SharedBarriers& sb, int bits) {
  sb.abort = 1;
  atomicOr(p.status, bits);
}

// ------------------------------------------------------------------ producer
template <int D, int BN, int MODE>
__device__ void attn_producer(const CUtensorMap* mapQ, const CUtensorMap* mapK, const CUtensorMap* mapV,
                              const AttnParams& p, uint8_t* sQ, uint8_t* sK, uint8_t* sV, SharedBarriers& sb) {
  using C = AttnCfg<D, BN>;
  volatile int* abort = &sb.abort;
  int g = 0, n = 0, bad = 0;
  bool ok = true;
  for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    const int kvh = h / p.group;
    TileIter it = make_iter<BN, MODE>(p, b, kvh, qt);
    int kb, bits;
    if (!it.next(kb, bits)) {
      bad |= it.bad;
      continue;
    }
    const int qbuf = n & 1;
    if (n >= 2 && !mbar_wait(&sb.q_empty[qbuf], ((n >> 1) - 1) & 1, abort)) {
      ok = false;
      break;
    }
    mbar_arrive_expect_tx(&sb.q_full[qbuf], C::kQBytes);
    for (int i = 0; i < C::kBoxes; ++i)
      tma_load_3d(sQ + qbuf * C::kQBytes + i * 128 * 128, mapQ, &sb.q_full[qbuf], 64 * i, qt * 128,
                  b * p.n_heads + h);
    ++n;
    do {
      const int s = g % C::kStages;
      if (g >= C::kStages && !mbar_wait(&sb.kv_empty[s], ((g / C::kStages) - 1) & 1, abort)) {
        ok = false;
        break;
      }
      const int z = b * p.n_kv_heads + kvh;
      mbar_arrive_expect_tx(&sb.k_full[s], C::kKVBytes);
      for (int i = 0; i < C::kBoxes; ++i)
        tma_load_3d(sK + s * C::kKVBytes + i * BN * 128, mapK, &sb.k_full[s], 64 * i, kb * BN, z);
      mbar_arrive_expect_tx(&sb.v_full[s], C::kKVBytes);
      for (int i = 0; i < C::kBoxes; ++i)
        tma_load_3d(sV + s * C::kKVBytes + i * BN * 128, mapV, &sb.v_full[s], 64 * i, kb * BN, z);
      ++g;
    } while (it.next(kb, bits));
    bad |= it.bad;
  }
  if (bad) atomicOr(p.status, kStatusBadSupport);
  if (!ok) {
    raise_status(p, sb, kStatusTimeout);
    // Let every copy already issued land before the CTA's shared memory is
    // released.
    int never = 0;
    for (int t = max(0, g - C::kStages); t < g; ++t) {
      mbar_wait(&sb.k_full[t % C::kStages], (t / C::kStages) & 1, &never);
      mbar_wait(&sb.v_full[t % C::kStages], (t / C::kStages) & 1, &never);
    }
    for (int m = max(0, n - 2); m < n; ++m) mbar_wait(&sb.q_full[m & 1], (m >> 1) & 1, &never);
  }
}

// ---------------------------------------------------------------- MMA issuer
template <int D, int BN>
__device__ __forceinline__ bool issue_pv(int t, bool first, uint32_t tmem, uint8_t* sP, uint8_t* sV,
                                         SharedBarriers& sb) {
  using C = AttnCfg<D, BN>;
  volatile int* abort = &sb.abort;
  if (!mbar_wait(&sb.p_full, t & 1, abort)) return false;
  const int s = t % C::kStages;
  if (!mbar_wait(&sb.v_full[s], (t / C::kStages) & 1, abort)) return false;
  tc_fence_after_sync();
  constexpr uint32_t idesc = idesc_bf16_f32(128, D, false, true);
  const uint32_t p_base = smem_u32(sP);
  const uint32_t v_base = smem_u32(sV + s * C::kKVBytes);
#pragma unroll
  for (int kk = 0; kk < BN / 16; ++kk) {
    const uint64_t a = smem_desc_sw128(p_base + (kk / 4) * 16384 + (kk % 4) * 32, 16, 1024);
    const uint64_t bdesc = smem_desc_sw128(v_base + kk * 2048, BN * 128, 1024);
    umma_bf16_ss(tmem + C::kTmemO, a, bdesc, idesc, (first && kk == 0) ? 0u : 1u);
  }
  umma_commit(&sb.kv_empty[s]);
  umma_commit(&sb.o_full);
  return true;
}

template <int D, int BN, int MODE>
__device__ void attn_mma(const AttnParams& p, uint32_t tmem, uint8_t* sQ, uint8_t* sK, uint8_t* sV, uint8_t* sP,
                         SharedBarriers& sb) {
  using C = AttnCfg<D, BN>;
  volatile int* abort = &sb.abort;
  constexpr uint32_t idesc_s = idesc_bf16_f32(128, BN, false, false);
  int g = 0, n = 0;
  bool ok = true;
  for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    TileIter it = make_iter<BN, MODE>(p, b, h / p.group, qt);
    int kb, bits;
    if (!it.next(kb, bits)) continue;
    const int qbuf = n & 1;
    if (!mbar_wait(&sb.q_full[qbuf], (n >> 1) & 1, abort)) {
      ok = false;
      break;
    }
    ++n;
    const uint32_t q_base = smem_u32(sQ + qbuf * C::kQBytes);
    int j = 0;
    bool more;
    do {
      const int s = g % C::kStages;
      if (!mbar_wait(&sb.k_full[s], (g / C::kStages) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint32_t k_base = smem_u32(sK + s * C::kKVBytes);
      const uint32_t s_tmem = tmem + (uint32_t)((g & 1) * BN);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t a = smem_desc_sw128(q_base + (kk / 4) * 16384 + (kk % 4) * 32, 16, 1024);
        const uint64_t bdesc = smem_desc_sw128(k_base + (kk / 4) * (BN * 128) + (kk % 4) * 32, 16, 1024);
        umma_bf16_ss(s_tmem, a, bdesc, idesc_s, kk > 0 ? 1u : 0u);
      }
      umma_commit(&sb.s_full[g & 1]);
      more = it.next(kb, bits);
      if (!more) umma_commit(&sb.q_empty[qbuf]);
      if (j > 0 && !issue_pv<D, BN>(g - 1, j == 1, tmem, sP, sV, sb)) {
        ok = false;
        break;
      }
      ++g;
      ++j;
    } while (more);
    if (ok && !issue_pv<D, BN>(g - 1, j == 1, tmem, sP, sV, sb)) ok = false;
  }
  if (!ok) raise_status(p, sb, kStatusTimeout);
  // Every MMA issued must have completed before TMEM is released.
  umma_commit(&sb.mma_done);
  int never = 0;
  mbar_wait(&sb.mma_done, 0, &never);
}

// ------------------------------------------------------------------- softmax
template <int D, int BN, int MODE>
__device__ void attn_softmax(const AttnParams& p, uint32_t tmem, uint8_t* sP, SharedBarriers& sb) {
  using C = AttnCfg<D, BN>;
  volatile int* abort = &sb.abort;
  const int r = threadIdx.x;  // query row within the tile, 0..127
  const int warp = r >> 5, lane = r & 31;
  const uint32_t lane_tmem = tmem + ((uint32_t)(warp * 32) << 16);
  const uint32_t p_base = smem_u32(sP);
  constexpr float kRescaleThreshold = 8.0f;  // log2 units: P stays <= 256
  int g = 0, epi_phase = 0;
  bool ok = true;
  for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    TileIter it = make_iter<BN, MODE>(p, b, h / p.group, qt);
    const int row = qt * 128 + r;
    const int half_bit = (BN == 64) ? (1 << (r >> 6)) : 1;
    float m_ref = -INFINITY, l = 0.0f;
    int j = 0, kb, bits, last_kb = -1;
    while (it.next(kb, bits)) {
      last_kb = kb;
      const int sbuf = g & 1;
      if (!warp_wait(&sb.s_full[sbuf], (g >> 1) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      float s[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(lane_tmem + sbuf * BN + 32 * c, v);
        tmem_ld_wait(v);
#pragma unroll
        for (int e = 0; e < 32; ++e) s[32 * c + e] = __uint_as_float(v[e]);
      }
      const int k0 = kb * BN;
      if (!(bits & half_bit)) {
#pragma unroll
        for (int c = 0; c < BN; ++c) s[c] = -INFINITY;
      } else if (k0 + BN - 1 > row) {
        const int lim = row - k0;  // keys k0 + c with c > lim are in the future
#pragma unroll
        for (int c = 0; c < BN; ++c) s[c] = (c > lim) ? -INFINITY : s[c];
      }
      float mx8[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) mx8[e] = s[e];
#pragma unroll
      for (int c = 8; c < BN; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], s[c]);
      const float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                             fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      const float m_tile = mx * p.scale_log2;
      float alpha = 1.0f;
      bool rescale = false;
      if (m_tile > m_ref + kRescaleThreshold) {
        alpha = ex2_approx(m_ref - m_tile);
        rescale = (m_ref != -INFINITY);
        m_ref = m_tile;
        l *= alpha;
      }
      const float m_use = (m_ref == -INFINITY) ? 0.0f : m_ref;
      float sum8[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) sum8[e] = 0.0f;
#pragma unroll
      for (int c = 0; c < BN; ++c) {
        s[c] = ex2_approx(fmaf(s[c], p.scale_log2, -m_use));
        sum8[c & 7] += s[c];
      }
      const float rowsum = ((sum8[0] + sum8[1]) + (sum8[2] + sum8[3])) + ((sum8[4] + sum8[5]) + (sum8[6] + sum8[7]));
      l += rowsum;
      if (MODE == kDenseMass)
        p.scratch[((size_t)blockIdx.x * p.n_blocks + kb) * 128 + r] =
            rowsum > 0.0f ? m_ref + lg2_approx(rowsum) : -INFINITY;
      // The previous tile's P V must be complete before O is rescaled and the
      // P buffer is overwritten.
      if (g > 0) {
        if (!warp_wait(&sb.o_full, (g - 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
      }
      // tcgen05.ld/st are warp-collective: the warp rescales together, lanes
      // whose max did not move use a factor of 1.
      if (j > 0 && __any_sync(0xffffffffu, rescale)) {
        const float f = rescale ? alpha : 1.0f;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(lane_tmem + C::kTmemO + 32 * c, v);
          tmem_ld_wait(v);
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * f);
          tmem_st_32x32b_x32(lane_tmem + C::kTmemO + 32 * c, v);
        }
        tmem_st_wait();
      }
#pragma unroll
      for (int c8 = 0; c8 < BN / 8; ++c8) {
        const uint32_t w0 = pack_bf16x2(s[8 * c8 + 0], s[8 * c8 + 1]);
        const uint32_t w1 = pack_bf16x2(s[8 * c8 + 2], s[8 * c8 + 3]);
        const uint32_t w2 = pack_bf16x2(s[8 * c8 + 4], s[8 * c8 + 5]);
        const uint32_t w3 = pack_bf16x2(s[8 * c8 + 6], s[8 * c8 + 7]);
        const uint32_t addr = p_base + (c8 / 8) * 16384 + r * 128 + (((c8 % 8) ^ (r & 7)) << 4);
        st_shared_v4(addr, w0, w1, w2, w3);
      }
      fence_proxy_async_smem();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sb.p_full);
      ++g;
      ++j;
    }
    if (!ok) break;
    // ---- epilogue: O / l
    if (j > 0) {
      if (!warp_wait(&sb.o_full, (g - 1) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
    }
    const float inv_l = l > 0.0f ? 1.0f / l : 0.0f;
    __nv_bfloat16* orow = p.O + ((size_t)(b * p.n_heads + h) * p.seqlen + row) * D;
#pragma unroll
    for (int c = 0; c < D / 32; ++c) {
      uint32_t v[32];
      if (j > 0) {
        tmem_ld_32x32b_x32(lane_tmem + C::kTmemO + 32 * c, v);
        tmem_ld_wait(v);
      } else {
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] = 0u;
      }
      uint32_t w[16];
#pragma unroll
      for (int e = 0; e < 16; ++e)
        w[e] = pack_bf16x2(__uint_as_float(v[2 * e]) * inv_l, __uint_as_float(v[2 * e + 1]) * inv_l);
      if (row < p.seqlen) {
        uint4* dst = reinterpret_cast<uint4*>(orow + 32 * c);
#pragma unroll
        for (int e = 0; e < 4; ++e) dst[e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
      }
    }
    // ---- epilogue: block mass (Eq. 5)
    if (MODE == kDenseMass) {
      float* red = reinterpret_cast<float*>(sP);  // every P V of this unit is complete
      const float lse = m_ref + lg2_approx(l);
      const int n_kt = last_kb + 1;
      for (int t = 0; t < n_kt; ++t) {
        const float lc = p.scratch[((size_t)blockIdx.x * p.n_blocks + t) * 128 + r];
        float v = (row < p.seqlen) ? ex2_approx(lc - lse) : 0.0f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (lane == 0) red[warp * p.n_blocks + t] = v;
      }
      mbar_arrive(&sb.epi);
      if (!warp_wait(&sb.epi, epi_phase & 1, abort)) {
        ok = false;
        break;
      }
      ++epi_phase;
      constexpr int kHalves = 128 / BN;
      const float inv_b = 1.0f / (float)BN;
      for (int e = r; e < kHalves * p.n_blocks; e += 128) {
        const int hf = e / p.n_blocks, t = e % p.n_blocks;
        const int qblock = qt * kHalves + hf;
        if (qblock >= p.n_blocks) continue;
        float* out = p.blockmass + ((size_t)(b * p.n_heads + h) * p.n_blocks + qblock) * p.n_blocks + t;
        if (t < n_kt) {
          float sum;
          if (BN == 128)
            sum = (red[0 * p.n_blocks + t] + red[1 * p.n_blocks + t]) +
                  (red[2 * p.n_blocks + t] + red[3 * p.n_blocks + t]);
          else
            sum = red[(2 * hf) * p.n_blocks + t] + red[(2 * hf + 1) * p.n_blocks + t];
          sum *= inv_b;
          *out = (p.step == 0) ? sum : *out + sum;
        } else if (p.step == 0) {
          *out = 0.0f;
        }
      }
      // `red` aliases the P tile, which the next unit overwrites.
      mbar_arrive(&sb.epi);
      if (!warp_wait(&sb.epi, epi_phase & 1, abort)) {
        ok = false;
        break;
      }
      ++epi_phase;
    }
  }
  if (!ok) raise_status(p, sb, kStatusTimeout);
}

// -------------------------------------------------------------------- kernel
template <int D, int BN, int MODE>
__global__ void __launch_bounds__(192, 1)
    attn_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                const __grid_constant__ CUtensorMap mapV, const AttnParams p) {
  using C = AttnCfg<D, BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + 2 * C::kQBytes;
  uint8_t* sV = sK + C::kStages * C::kKVBytes;
  uint8_t* sP = sV + C::kStages * C::kKVBytes;
  __shared__ SharedBarriers sb;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    sb.abort = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sb.q_full[i], 1);
      mbar_init(&sb.q_empty[i], 1);
      mbar_init(&sb.s_full[i], 1);
    }
    for (int i = 0; i < C::kStages; ++i) {
      mbar_init(&sb.k_full[i], 1);
      mbar_init(&sb.v_full[i], 1);
      mbar_init(&sb.kv_empty[i], 1);
    }
    mbar_init(&sb.p_full, 4);
    mbar_init(&sb.o_full, 1);
    mbar_init(&sb.mma_done, 1);
    mbar_init(&sb.epi, 128);
    fence_mbar_init();
  }
  if (warp == 4 && lane == 0) {
    tma_prefetch_map(&mapQ);
    tma_prefetch_map(&mapK);
    tma_prefetch_map(&mapV);
  }
  if (warp == 5) {
    tmem_alloc(&sb.tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sb.tmem_base;

  if (warp < 4) {
    attn_softmax<D, BN, MODE>(p, tmem, sP, sb);
  } else if (warp == 4) {
    if (lane == 0) attn_producer<D, BN, MODE>(&mapQ, &mapK, &mapV, p, sQ, sK, sV, sb);
  } else {
    if (lane == 0) attn_mma<D, BN, MODE>(p, tmem, sQ, sK, sV, sP, sb);
  }

  __syncwarp();
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after_sync();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int D, int BN, int MODE>
cudaError_t launch_attn_instance(const AttnLaunch& L) {
  using C = AttnCfg<D, BN>;
  auto kern = attn_kernel<D, BN, MODE>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemLaunch);
  if (e != cudaSuccess) return e;
  kern<<<L.grid, C::kThreads, C::kSmemLaunch, L.stream>>>(L.mapQ, L.mapK, L.mapV, L.p);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_attn_for_dim(int block, int mode, const AttnLaunch& L) {
  if (block == 128) {
    if (mode == kDense) return launch_attn_instance<D, 128, kDense>(L);
    if (mode == kDenseMass) return launch_attn_instance<D, 128, kDenseMass>(L);
    return launch_attn_instance<D, 128, kSparse>(L);
  }
  if (mode == kDense) return launch_attn_instance<D, 64, kDense>(L);
  if (mode == kDenseMass) return launch_attn_instance<D, 64, kDenseMass>(L);
  return launch_attn_instance<D, 64, kSparse>(L);
}

}  // namespace wise
