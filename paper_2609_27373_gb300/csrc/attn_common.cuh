// Pieces shared by the attention kernels: the key-tile width, the tile
// schedule entries, the softmax arithmetic (log2-domain exponentials, row
// maxima), the iterator over a unit's key tiles (dense prefix or the merge of
// the support lists), unit decoding, TMEM row loads with the causal/support
// mask, and the bounded warp-wide wait.
#pragma once

#include <cuda_bf16.h>
#include <limits.h>
#include <stdint.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace wise {

// Key tiles are 128 keys wide whatever the block size: a tcgen05 MMA issued by
// one thread costs about the same issue time at N = 32, 64 or 128, so narrower
// tiles only waste tensor throughput.  Blocks of 32 or 64 are sub-blocks of a
// tile, selected per (query block, key block) by the tile's mask.
constexpr int kTileN = 128;

// Tile schedule rings.  Entry = {key tile | mask << 16, unit, flags, tile
// index within its unit} (for the end marker: {0, 0, kEntEnd, number of
// tiles}).  With S = 128 / block query blocks per query tile and key blocks
// per key tile, bit qi * S + ki of the mask says that query block qi of the
// tile attends key block ki of the key tile.  Flag bits 8 and up hold the
// index of the unit among this CTA's units with tiles.
constexpr int kSchedSlots = 16;  // per ring
constexpr int kEntFirst = 4;     // first tile of its unit
constexpr int kEntLast = 8;      // last tile of its unit
constexpr int kEntEmpty = 16;    // unit without tiles (its output rows are zero)
constexpr int kEntEnd = 32;      // no more units for this CTA
constexpr int kEntUnitShift = 8;
constexpr int kMmaRing = 2;  // ring of the two MMA threads

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

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Maximum of n values with a tree of three-input max operations.
template <int N>
__device__ __forceinline__ float row_max(const float (&s)[N]) {
  float m[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) m[e] = s[e];
#pragma unroll
  for (int c = 8; c + 1 < N; c += 16) {
#pragma unroll
    for (int e = 0; e < 8; ++e) m[e] = fmax3(m[e], s[c + e], (c + 8 + e < N) ? s[c + 8 + e] : s[c + e]);
  }
  return fmaxf(fmax3(m[0], m[1], m[2]), fmax3(fmax3(m[3], m[4], m[5]), m[6], m[7]));
}

// p = 2^(s * scale - shift) in place, two elements per packed FMA; returns
// the sum of p.
template <int N>
__device__ __forceinline__ float exp2_scaled(float (&s)[N], float scale, float shift) {
  const float2 sc = make_float2(scale, scale), sh = make_float2(-shift, -shift);
  float2 acc[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) acc[e] = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int c = 0; c < N; c += 2) {
    const float2 x = __ffma2_rn(make_float2(s[c], s[c + 1]), sc, sh);
    const float2 y = make_float2(ex2_approx(x.x), ex2_approx(x.y));
    s[c] = y.x;
    s[c + 1] = y.y;
    acc[(c / 2) & 3] = __fadd2_rn(acc[(c / 2) & 3], y);
  }
  const float2 b = __fadd2_rn(__fadd2_rn(acc[0], acc[1]), __fadd2_rn(acc[2], acc[3]));
  return b.x + b.y;
}

// exp2_scaled that also returns the sums of the S column groups of N / S
// columns (the key sub-blocks of a tile), for the block masses; S = 2 or 4.
template <int N, int S>
__device__ __forceinline__ float exp2_scaled_groups(float (&s)[N], float scale, float shift, float (&g)[S]) {
  static_assert(S == 2 || S == 4, "groups");
  constexpr int kChains = 4 / S;  // independent accumulation chains per group
  constexpr int kCols = N / S;
  const float2 sc = make_float2(scale, scale), sh = make_float2(-shift, -shift);
  float2 acc[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) acc[e] = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int c = 0; c < N; c += 2) {
    const float2 x = __ffma2_rn(make_float2(s[c], s[c + 1]), sc, sh);
    const float2 y = make_float2(ex2_approx(x.x), ex2_approx(x.y));
    s[c] = y.x;
    s[c + 1] = y.y;
    const int a = (c / kCols) * kChains + (c / 2) % kChains;
    acc[a] = __fadd2_rn(acc[a], y);
  }
  float total = 0.0f;
#pragma unroll
  for (int k = 0; k < S; ++k) {
    float2 t = acc[k * kChains];
#pragma unroll
    for (int ch = 1; ch < kChains; ++ch) t = __fadd2_rn(t, acc[k * kChains + ch]);
    g[k] = t.x + t.y;
    total += g[k];
  }
  return total;
}

// Column sums over the 32 lanes of a warp: v[i] holds this lane's value of
// column i; returns the sum of column `lane`.  Each step exchanges half of
// the remaining columns with the lane `o` away (o = 16, 8, 4, 2, 1), 31
// shuffles in all.  The additions pair the lanes exactly as a butterfly
// reduction with the same offsets does, so every column sum is the same bit
// for bit.
__device__ __forceinline__ float warp_column_sums(float (&v)[32], int lane) {
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float send = upper ? v[i] : v[i + o];
      const float keep = upper ? v[i + o] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
    }
  }
  return v[0];
}

// Key tiles of one unit in ascending order, with their sub-block masks
// (S = 128 / BLK).  Dense: tiles 0..last, every sub-block (the causal limit is
// applied per row).  Sparse: the merge of the support lists of the unit's S
// query blocks; key block kb lies in key tile kb / S.  Entries that are
// negative, beyond their query block, or not strictly ascending are skipped
// and flagged in `bad`.  Fields a variant does not use are never touched, so
// they cost no registers.
template <int BLK, int MODE>
struct TileIter {
  static constexpr int S = kTileN / BLK;
  int cur, last;             // dense
  const int32_t* l0;         // sparse: list of query block q0; list q at l0 + q * cap
  int cap, q0;
  int pos[S];                // list q: entries read (low 16 bits) and count (high 16 bits); cap < 2^16
  int pend[S];               // next entry of list q (the last one accepted), INT_MAX when done
  int bad;

  // Next valid entry of list q after pend[q]: in [0, q0 + q] and above it.
  __device__ __forceinline__ int pull(int q) {
    const int prev = pend[q];
    while ((pos[q] & 0xFFFF) < (pos[q] >> 16)) {
      const int v = __ldg(l0 + (size_t)q * cap + (pos[q] & 0xFFFF));
      ++pos[q];
      if (v >= 0 && v <= q0 + q && v > prev) return v;
      bad = 1;
    }
    return INT_MAX;
  }

  __device__ __forceinline__ bool next(int& kt, uint32_t& mask) {
    if constexpr (MODE != kSparse) {
      if (cur > last) return false;
      kt = cur++;
      mask = S == 1 ? 1u : S == 2 ? 0xFu : 0xFFFFu;
      return true;
    } else {
      int lo = pend[0];
#pragma unroll
      for (int q = 1; q < S; ++q) lo = min(lo, pend[q]);
      if (lo == INT_MAX) return false;
      kt = lo / S;
      mask = 0;
#pragma unroll
      for (int q = 0; q < S; ++q) {
        while (pend[q] != INT_MAX && pend[q] / S == kt) {
          mask |= 1u << (q * S + pend[q] % S);
          pend[q] = pull(q);
        }
      }
      return true;
    }
  }
};

__device__ __forceinline__ int clamp_count(int n, int cap, int& bad) {
  if (n < 0 || n > cap) {
    bad = 1;
    return n < 0 ? 0 : cap;
  }
  return n;
}

template <int BLK, int MODE>
__device__ __forceinline__ TileIter<BLK, MODE> make_iter(const AttnParams& p, int b, int kvh, int qt) {
  TileIter<BLK, MODE> it;
  it.bad = 0;
  if constexpr (MODE != kSparse) {
    it.cur = 0;
    const int last_row = min(qt * 128 + 127, p.seqlen - 1);
    it.last = last_row / kTileN;
  } else {
    constexpr int S = TileIter<BLK, MODE>::S;
    const int q0 = qt * S;
    const size_t row0 = ((size_t)b * p.n_kv_heads + kvh) * p.n_blocks + q0;
    it.l0 = p.idx + row0 * p.cap;
    it.cap = p.cap;
    it.q0 = q0;
#pragma unroll
    for (int q = 0; q < S; ++q) {
      it.pos[q] = ((q0 + q < p.n_blocks) ? clamp_count(__ldg(p.counts + row0 + q), p.cap, it.bad) : 0) << 16;
      it.pend[q] = -1;
    }
#pragma unroll
    for (int q = 0; q < S; ++q) it.pend[q] = it.pull(q);
  }
  return it;
}

// Unit u -> (batch, head, query tile).  Units are numbered by decreasing
// causal length (the grid deals them out in a snake order that evens out the
// per-CTA sums).  With group_heads > 0 the (batch, head) pairs are taken in
// groups of group_heads consecutive ones (whole kv-head groups), all units of
// a group before the next, so that the K and V of a group stay in L2 while
// all its query tiles read them.
__device__ __forceinline__ void decode_unit(const AttnParams& p, int u, int& b, int& h, int& qt) {
  const int bh_count = p.batch * p.n_heads;
  int bh;
  if (p.group_heads > 0) {
    const int per_group = p.group_heads * p.n_qtiles;
    const int g = u / per_group, v = u - g * per_group;
    const int gh = min(p.group_heads, bh_count - g * p.group_heads);  // the last group may be smaller
    qt = p.n_qtiles - 1 - v / gh;
    bh = g * p.group_heads + v % gh;
  } else {
    qt = p.n_qtiles - 1 - u / bh_count;
    bh = u % bh_count;
  }
  b = bh / p.n_heads;
  h = bh % p.n_heads;
}

// mbar_wait whose outcome is the same for every lane of the warp (all lanes
// must call it together): a lane that gave up makes the whole warp give up.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort,
                                          uint64_t limit_ns = kWaitLimitNs) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, limit_ns));
}

__device__ __forceinline__ void raise_status(const AttnParams& p, int* abort, int bits) {
  *reinterpret_cast<volatile int*>(abort) = 1;
  atomicOr(p.status, bits);
}

// Loads N consecutive 32-bit TMEM columns of this thread's lane (N = 64, 96
// or 128: 32-column loads issued together, one wait).
template <int N>
__device__ __forceinline__ void tmem_load_row(uint32_t addr, float (&x)[N]) {
  static_assert(N == 64 || N == 96 || N == 128, "row width");
  uint32_t va[32], vb[32], vc[32], vd[32];
  tmem_ld_32x32b_x32(addr, va);
  tmem_ld_32x32b_x32(addr + 32, vb);
  if constexpr (N >= 96) tmem_ld_32x32b_x32(addr + 64, vc);
  if constexpr (N == 128) tmem_ld_32x32b_x32(addr + 96, vd);
  tmem_ld_wait(va, vb);  // completes every load issued above
  if constexpr (N >= 96) reg_tie(vc);
  if constexpr (N == 128) reg_tie(vd);
#pragma unroll
  for (int e = 0; e < 32; ++e) {
    x[e] = __uint_as_float(va[e]);
    x[32 + e] = __uint_as_float(vb[e]);
    if constexpr (N >= 96) x[64 + e] = __uint_as_float(vc[e]);
    if constexpr (N == 128) x[96 + e] = __uint_as_float(vd[e]);
  }
}

// Applies the causal / support masks to this thread's row of an S tile
// (kTileN columns): column c of key sub-block k = c / BLK is kept if
// bit k of `sub` is set and c <= lim (keys with c > lim are in the future of
// this row).
template <int BLK>
__device__ __forceinline__ void mask_s_row(float (&s)[kTileN], uint32_t sub, int lim) {
  constexpr int S = kTileN / BLK;
  if (sub != (1u << S) - 1u || lim < kTileN - 1) {
    // Per sub-block limit: lim where the row attends the sub-block, else the
    // column before it, so that a single compare masks the column.
    int lim_k[S];
#pragma unroll
    for (int k = 0; k < S; ++k) lim_k[k] = ((sub >> k) & 1u) ? lim : k * BLK - 1;
#pragma unroll
    for (int c = 0; c < kTileN; ++c) s[c] = (c > lim_k[c / BLK]) ? -INFINITY : s[c];
  }
}

// Loads this thread's row of an S tile and applies the masks.
template <int BLK>
__device__ __forceinline__ void load_s_row(uint32_t addr, float (&s)[kTileN], uint32_t sub, int lim) {
  tmem_load_row<kTileN>(addr, s);
  mask_s_row<BLK>(s, sub, lim);
}

}  // namespace wise
