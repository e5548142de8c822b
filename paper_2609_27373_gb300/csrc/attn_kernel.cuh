// Causal flash attention on tcgen05 tensor cores, in three variants:
//   kDense      O = softmax(Q K^T * scale + M) V                  (Eq. 2)
//   kDenseMass  the same, plus the block attention mass of the step (Eq. 5)
//               accumulated into blockmass
//   kSparse     key blocks restricted to the selected support      (Eqs. 7-8)
//
// Work decomposition.  A unit is one 128-row query tile of one (batch, head);
// units are numbered in order of decreasing causal length, and the
// persistent grid (one CTA per SM) hands CTA c the units c, c + grid, ...
// Each unit walks its list of key tiles (BN = block keys each): every tile of
// the causal prefix (dense), or the blocks of the support (sparse; with block
// 64 a query tile covers two query blocks and walks the union of their lists,
// masking per half).
//
// Both products run with the A operand in tensor memory, because a tcgen05
// MMA that reads both operands from shared memory is limited by the shared
// memory read rate to about half the tensor peak (measured: 118 clk per
// M128/N128/K16 step with both operands in shared memory, 66 clk with A in
// TMEM):
//   S = Q K^T    Q copied once per unit from shared memory into TMEM, K
//                from shared memory (K-major);
//   O += P V     P written by the softmax into TMEM, V from shared memory
//                (MN-major).
// TMEM (512 columns): Q double-buffered across units (2 x 64 columns), S
// double-buffered across tiles (2 x 128 columns, P overwrites the first BN/2
// columns of its S), O (128 columns).
//
// Warp roles (352 threads):
//   warps 0-3 and 4-7  two softmax warpgroups.  Thread t of warpgroup h owns
//              query row t (= TMEM lane t), key columns [h BN/2, (h+1) BN/2)
//              of every S tile and output columns [h D/2, (h+1) D/2) of O.
//              Per tile it loads its half row of S, exchanges the half-row
//              maximum with its partner thread (bounded mbarrier), keeps the
//              running max and its half of the row sum (online softmax in the
//              log2 domain; O is rescaled only when the max grows by more than
//              2^8), and writes its half of P into TMEM.  Per unit it copies
//              the next unit's Q into TMEM and runs the epilogue: O / l to
//              global memory and, for kDenseMass, the block masses.
//   warp 8     TMA producer: K tiles into a ring of kRingK entries and V tiles
//              into a ring of kRingV entries, in the order K(0), K(1), V(0),
//              K(2), V(1), ...
//   warp 9     S issuer: S(j) = Q K(j)^T into S buffer j & 1, one tile ahead
//              of the softmax.
//   warp 10    P V issuer: O += P(j) V(j) once the softmax has written P(j).
//   A tcgen05.mma issue blocks its thread while the tensor core drains the
//   previous instructions, so the two products are issued from two threads:
//   each thread's barrier checks overlap the other's issue and the tensor
//   core stays fed.  S(j) reuses the buffer of P(j-2); the P V thread commits
//   buf_free[b] after each P V so that the S thread can wait for it.
//
#pragma once

#include <cuda_bf16.h>
#include <limits.h>
#include <stdint.h>

#include <type_traits>

#include "internal.cuh"
#include "ptx.cuh"

// Pairs (of every 8) of softmax exponentials evaluated on the FMA pipe
// instead of MUFU (0 = all on MUFU).
#ifndef WISE_EMU_PAIRS
#define WISE_EMU_PAIRS 0
#endif

namespace wise {

template <int D, int BN>
struct AttnCfg {
  static constexpr int kBoxes = (D + 63) / 64;          // 64-column TMA boxes per row tile
  static constexpr int kQBytes = kBoxes * 128 * 128;    // one 128-row Q tile (staging)
  static constexpr int kKVBytes = kBoxes * BN * 128;    // one BN-row K or V tile (one ring entry)
  // Dynamic shared memory available after the 1024-byte alignment slack and
  // the static barriers and exchange buffers.
  static constexpr int kBudget = 227 * 1024 - 1024 - 2560;
  static constexpr int kRingFit = (kBudget - kQBytes) / kKVBytes;
  static constexpr int kRing = kRingFit > 12 ? 12 : kRingFit;
  static constexpr int kRingK = (kRing + 1) / 2;  // K tiles (consumed by S)
  static constexpr int kRingV = kRing / 2;        // V tiles (consumed by P V)
  static constexpr int kSmemBytes = kQBytes + kRing * kKVBytes + 1024;
  // At least 116 KB so that a single CTA resides per SM (it owns all 512
  // TMEM columns).
  static constexpr int kSmemLaunch = kSmemBytes > 116 * 1024 ? kSmemBytes : 116 * 1024;
  static constexpr uint32_t kTmemQ = 0;       // two Q buffers
  static constexpr uint32_t kTmemQCols = 64;  // 128 bf16 of Q per row
  static constexpr uint32_t kTmemS = 128;     // two S/P buffers
  static constexpr uint32_t kTmemSCols = 128;
  static constexpr uint32_t kTmemO = 384;     // O accumulator
  static constexpr uint32_t kTmemCols = 512;
  static constexpr int kThreads = 352;
  static constexpr int kProducerWarp = 8;
  static constexpr int kMmaSWarp = 9;   // issues S = Q K^T, owns the TMEM allocation
  static constexpr int kMmaPVWarp = 10; // issues O += P V
  static_assert(kRingV >= 1 && kRingK >= 2, "shared memory budget");
  static_assert(BN <= 128 && D <= 128, "TMEM budget");
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

// 2^x for a pair of values on the FMA and integer pipes, leaving the MUFU
// unit to the other exponentials (the softmax is otherwise bound by MUFU
// throughput, 16 ex2 per clock per SM).  Cody-Waite style reduction: adding
// 1.5 * 2^23 rounds x to the nearest integer n (which also appears in the low
// mantissa bits of the sum), f = x - n lies in [-1/2, 1/2], 2^f is a degree-3
// polynomial fitted here to minimise the maximum relative error on that
// interval (7.5e-5 with fp32 Horner evaluation), and n is added to the
// exponent field.  Inputs are clamped to [-126, 64] (so the exponent field
// cannot wrap); the results feed bf16 probabilities (relative precision
// 3.9e-3).  Masked inputs (-inf) need exp2_scaled's masked path for an exact 0.
__device__ __forceinline__ float2 exp2_poly2(float2 x) {
  constexpr float kRound = 12582912.0f;  // 1.5 * 2^23
  const float2 xc = make_float2(fminf(fmaxf(x.x, -126.0f), 64.0f), fminf(fmaxf(x.y, -126.0f), 64.0f));
  const float2 t = __fadd2_rn(xc, make_float2(kRound, kRound));
  const float2 n = __fadd2_rn(t, make_float2(-kRound, -kRound));
  const float2 f = __fadd2_rn(xc, make_float2(-n.x, -n.y));
  float2 q = __ffma2_rn(make_float2(5.517166853e-02f, 5.517166853e-02f), f,
                        make_float2(2.426111251e-01f, 2.426111251e-01f));
  q = __ffma2_rn(q, f, make_float2(6.932609677e-01f, 6.932609677e-01f));
  q = __ffma2_rn(q, f, make_float2(9.999280572e-01f, 9.999280572e-01f));
  // The rounded integer sits in the low mantissa bits of t: shift it into the
  // exponent field (the constant part of t's bits cancels modulo 2^32).
  constexpr int kBias = (int)(0x4B400000u << 23);
  return make_float2(__int_as_float(__float_as_int(q.x) + (__float_as_int(t.x) << 23) - kBias),
                     __int_as_float(__float_as_int(q.y) + (__float_as_int(t.y) << 23) - kBias));
}

// p = 2^(s * scale - shift) in place, two elements per packed FMA; returns
// the sum of p.  kEmu of every 8 pairs use exp2_poly2, the rest MUFU ex2.
// With `masked` (the row has masked keys in this tile) emulated results of
// inputs below -126 are forced to exactly 0, as ex2 gives for -inf.
template <int kEmu, int N>
__device__ __forceinline__ float exp2_scaled(float (&s)[N], float scale, float shift, bool masked) {
  const float2 sc = make_float2(scale, scale), sh = make_float2(-shift, -shift);
  float2 acc[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) acc[e] = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int c = 0; c < N; c += 2) {
    const float2 x = __ffma2_rn(make_float2(s[c], s[c + 1]), sc, sh);
    float2 y;
    if ((c / 2) % 8 < kEmu) {
      y = exp2_poly2(x);
      if (masked) {
        y.x = x.x < -126.0f ? 0.0f : y.x;
        y.y = x.y < -126.0f ? 0.0f : y.y;
      }
    } else {
      y.x = ex2_approx(x.x);
      y.y = ex2_approx(x.y);
    }
    s[c] = y.x;
    s[c + 1] = y.y;
    acc[(c / 2) & 3] = __fadd2_rn(acc[(c / 2) & 3], y);
  }
  const float2 b = __fadd2_rn(__fadd2_rn(acc[0], acc[1]), __fadd2_rn(acc[2], acc[3]));
  return b.x + b.y;
}

// Key tiles of one unit in ascending order.  Dense: 0..last.  Sparse: the
// support list of the unit's query block (block 128), or the merge of the
// lists of its two query blocks (block 64); `bits` says which half of the
// 128 query rows may attend the tile.  Entries that are negative, beyond the
// query block, or not strictly ascending are skipped and flagged in `bad`.
// Fields a variant does not use are never touched, so they cost no registers.
template <int BN, int MODE>
struct TileIter {
  int cur, last;                                   // dense
  const int32_t* la;                               // sparse, first query block
  int na, ia, lima, preva, pend_a;
  const int32_t* lb;                               // sparse, second query block (block 64)
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
    if constexpr (MODE != kSparse) {
      if (cur > last) return false;
      kb = cur++;
      bits = 3;
      return true;
    } else if constexpr (BN == 128) {
      if (pend_a == INT_MAX) return false;
      kb = pend_a;
      bits = 1;
      pend_a = pull(la, na, ia, lima, preva);
      return true;
    } else {
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
__device__ __forceinline__ TileIter<BN, MODE> make_iter(const AttnParams& p, int b, int kvh, int qt) {
  TileIter<BN, MODE> it;
  it.bad = 0;
  if constexpr (MODE != kSparse) {
    it.cur = 0;
    const int last_row = min(qt * 128 + 127, p.seqlen - 1);
    it.last = last_row / BN;
  } else {
    constexpr int kQbPerTile = 128 / BN;
    const int q0 = qt * kQbPerTile;
    const size_t row0 = ((size_t)b * p.n_kv_heads + kvh) * p.n_blocks + q0;
    it.la = p.idx + row0 * p.cap;
    it.na = clamp_count(__ldg(p.counts + row0), p.cap, it.bad);
    it.ia = 0;
    it.lima = q0;
    it.preva = -1;
    it.pend_a = it.pull(it.la, it.na, it.ia, it.lima, it.preva);
    if constexpr (kQbPerTile == 2) {
      it.lb = p.idx + (row0 + 1) * p.cap;
      it.nb = (q0 + 1 < p.n_blocks) ? clamp_count(__ldg(p.counts + row0 + 1), p.cap, it.bad) : 0;
      it.ib = 0;
      it.limb = q0 + 1;
      it.prevb = -1;
      it.pend_b = it.pull(it.lb, it.nb, it.ib, it.limb, it.prevb);
    }
  }
  return it;
}

__device__ __forceinline__ void decode_unit(const AttnParams& p, int u, int& b, int& h, int& qt) {
  const int bh_count = p.batch * p.n_heads;
  qt = p.n_qtiles - 1 - u / bh_count;  // longest causal prefix first
  const int bh = u % bh_count;
  b = bh / p.n_heads;
  h = bh % p.n_heads;
}

// One key tile of the CTA's stream, as the producer and the MMA warp need it.
struct Tile {
  int kb;     // key block
  int z;      // batch * n_kv_heads + kv head (TMA outer coordinate of K and V)
  int first;  // first tile of its unit
};

// The tiles of one CTA, unit after unit (units without any tile skipped).
template <int BN, int MODE>
struct TileStream {
  int u, stride, z;
  TileIter<BN, MODE> it;
  int nkb, nfirst, have;
  int bad;

  __device__ __forceinline__ void open_next_unit(const AttnParams& p) {
    for (;;) {
      u += stride;
      if (u >= p.n_units) {
        have = 0;
        return;
      }
      int b, h, qt;
      decode_unit(p, u, b, h, qt);
      const int kvh = h / p.group;
      z = b * p.n_kv_heads + kvh;
      it = make_iter<BN, MODE>(p, b, kvh, qt);
      int bits;
      if (it.next(nkb, bits)) {
        nfirst = 1;
        have = 1;
        return;
      }
      bad |= it.bad;
    }
  }

  __device__ __forceinline__ void start(const AttnParams& p) {
    stride = gridDim.x;
    u = blockIdx.x - stride;
    bad = 0;
    open_next_unit(p);
  }

  __device__ __forceinline__ bool next(const AttnParams& p, Tile& t) {
    if (!have) return false;
    t.kb = nkb;
    t.z = z;
    t.first = nfirst;
    int bits;
    if (it.next(nkb, bits)) {
      nfirst = 0;
    } else {
      bad |= it.bad;
      open_next_unit(p);
    }
    return true;
  }
};

template <int RK, int RV>
struct SharedBarriers {
  uint64_t k_full[RK], k_empty[RK], v_full[RV], v_empty[RV];
  // Barriers that a thread may reach late (after the producing side has
  // already moved on by one item) exist once per buffer: a second completion
  // of the same barrier then needs work that the waiting thread itself has
  // not issued yet, so a parity wait can never skip a phase.
  uint64_t q_full;       // Q tile landed in the staging buffer (TMA)
  uint64_t q_tmem[2];    // Q copied into TMEM buffer b (8 softmax warps)
  uint64_t s_full[2];    // S buffer b written (S thread commit)
  uint64_t buf_free[2];  // P of buffer b consumed by its P V (P V thread commit)
  uint64_t p_full[2];    // P of buffer b written into TMEM (8 softmax warps)
  uint64_t o_full;       // a P V completed (P V thread commit)
  uint64_t xch;          // the two softmax halves exchanged row values (8 warps)
  uint64_t s_done, pv_done;
  float xbuf[2][2][128];  // [phase & 1][half][row]
  uint32_t tmem_base;
  int abort;
};

// mbar_wait whose outcome is the same for every lane of the warp (all lanes
// must call it together): a lane that gave up makes the whole warp give up.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

__device__ __forceinline__ void raise_status(const AttnParams& p, int* abort, int bits) {
  *reinterpret_cast<volatile int*>(abort) = 1;
  atomicOr(p.status, bits);
}

// ------------------------------------------------------------------ producer
template <int D, int BN, int MODE>
__device__ void attn_producer(const CUtensorMap* mapK, const CUtensorMap* mapV, const AttnParams& p, uint8_t* ring,
                              SharedBarriers<AttnCfg<D, BN>::kRingK, AttnCfg<D, BN>::kRingV>& sb) {
  using C = AttnCfg<D, BN>;
  constexpr int RK = C::kRingK, RV = C::kRingV;
  uint8_t* k_ring = ring;
  uint8_t* v_ring = ring + RK * C::kKVBytes;
  volatile int* abort = &sb.abort;
  TileStream<BN, MODE> st;
  st.start(p);
  int jk = 0, jv = 0;
  bool ok = true;
  auto load = [&](const CUtensorMap* map, uint8_t* base, uint64_t* full, uint64_t* empty, int R, int& j,
                  const Tile& t) -> bool {
    const int slot = j % R;
    if (j >= R && !mbar_wait(&empty[slot], ((j / R) - 1) & 1, abort)) return false;
    mbar_arrive_expect_tx(&full[slot], C::kKVBytes);
    for (int i = 0; i < C::kBoxes; ++i)
      tma_load_3d(base + slot * C::kKVBytes + i * BN * 128, map, &full[slot], 64 * i, t.kb * BN, t.z);
    ++j;
    return true;
  };
  Tile cur, nxt;
  bool have = st.next(p, cur);
  if (have && !load(mapK, k_ring, sb.k_full, sb.k_empty, RK, jk, cur)) ok = false;
  while (have && ok) {
    const bool more = st.next(p, nxt);
    if (more && !load(mapK, k_ring, sb.k_full, sb.k_empty, RK, jk, nxt)) {
      ok = false;
      break;
    }
    if (!load(mapV, v_ring, sb.v_full, sb.v_empty, RV, jv, cur)) {
      ok = false;
      break;
    }
    cur = nxt;
    have = more;
  }
  if (st.bad) atomicOr(p.status, kStatusBadSupport);
  if (!ok) {
    raise_status(p, &sb.abort, kStatusTimeout);
    // Let every copy already issued land before the CTA's shared memory is
    // released.
    int never = 0;
    for (int t = max(0, jk - RK); t < jk; ++t) mbar_wait(&sb.k_full[t % RK], (t / RK) & 1, &never);
    for (int t = max(0, jv - RV); t < jv; ++t) mbar_wait(&sb.v_full[t % RV], (t / RV) & 1, &never);
  }
}

// --------------------------------------------------------------- MMA issuers
template <int D, int BN, int MODE>
__device__ void attn_mma_s(const AttnParams& p, uint32_t tmem, uint8_t* ring,
                           SharedBarriers<AttnCfg<D, BN>::kRingK, AttnCfg<D, BN>::kRingV>& sb) {
  using C = AttnCfg<D, BN>;
  constexpr int RK = C::kRingK;
  volatile int* abort = &sb.abort;
  constexpr uint32_t idesc_s = idesc_bf16_f32(128, BN, false, false);
  TileStream<BN, MODE> st;
  st.start(p);
  int n_q = 0;
  uint32_t q_col = 0;  // TMEM column of the current unit's Q
  bool ok = true;
  Tile t;
  for (int j = 0; st.next(p, t); ++j) {
    if (t.first) {
      if (!mbar_wait(&sb.q_tmem[n_q & 1], (n_q >> 1) & 1, abort)) ok = false;
      q_col = C::kTmemQ + (n_q & 1) * C::kTmemQCols;
      ++n_q;
    }
    const int slot = j % RK;
    if (ok && !mbar_wait(&sb.k_full[slot], (j / RK) & 1, abort)) ok = false;
    // S(j) overwrites the buffer that held P(j-2).
    if (ok && j >= 2 && !mbar_wait(&sb.buf_free[j & 1], ((j >> 1) - 1) & 1, abort)) ok = false;
    if (!ok) break;
    tc_fence_after_sync();
    const uint32_t s_col = C::kTmemS + (j & 1) * C::kTmemSCols;
    const uint64_t b0 = smem_desc_sw128(smem_u32(ring + slot * C::kKVBytes), 16, 1024);
#pragma unroll 1
    for (int kk = 0; kk < D / 16; ++kk) {
      // K step kk: 8 TMEM columns of Q; shared-memory descriptors of later
      // steps differ only in the start address field (address >> 4).
      const uint32_t b_off = ((kk >> 2) * (BN * 128) + (kk & 3) * 32) >> 4;
      umma_bf16_ts(tmem + s_col, tmem + q_col + kk * 8, b0 + b_off, idesc_s, kk > 0 ? 1u : 0u);
    }
    umma_commit(&sb.s_full[j & 1]);
    umma_commit(&sb.k_empty[slot]);
  }
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
  // Every MMA issued must have completed before TMEM is released.
  umma_commit(&sb.s_done);
  int never = 0;
  mbar_wait(&sb.s_done, 0, &never);
}

template <int D, int BN, int MODE>
__device__ void attn_mma_pv(const AttnParams& p, uint32_t tmem, uint8_t* ring,
                            SharedBarriers<AttnCfg<D, BN>::kRingK, AttnCfg<D, BN>::kRingV>& sb) {
  using C = AttnCfg<D, BN>;
  constexpr int RK = C::kRingK, RV = C::kRingV;
  uint8_t* v_ring = ring + RK * C::kKVBytes;
  volatile int* abort = &sb.abort;
  constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);
  TileStream<BN, MODE> st;
  st.start(p);
  bool ok = true;
  Tile t;
  for (int j = 0; st.next(p, t); ++j) {
    const int slot = j % RV;
    if (!mbar_wait(&sb.p_full[j & 1], (j >> 1) & 1, abort)) ok = false;
    if (ok && !mbar_wait(&sb.v_full[slot], (j / RV) & 1, abort)) ok = false;
    if (!ok) break;
    tc_fence_after_sync();
    // P(j) sits in the first BN/2 columns of S buffer j & 1.
    const uint32_t p_col = C::kTmemS + (j & 1) * C::kTmemSCols;
    const uint64_t b0 = smem_desc_sw128(smem_u32(v_ring + slot * C::kKVBytes), BN * 128, 1024);
#pragma unroll 1
    for (int kk = 0; kk < BN / 16; ++kk)
      umma_bf16_ts(tmem + C::kTmemO, tmem + p_col + kk * 8, b0 + ((kk * 2048) >> 4), idesc_o,
                   (t.first && kk == 0) ? 0u : 1u);
    umma_commit(&sb.o_full);
    umma_commit(&sb.v_empty[slot]);
    umma_commit(&sb.buf_free[j & 1]);
  }
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
  umma_commit(&sb.pv_done);
  int never = 0;
  mbar_wait(&sb.pv_done, 0, &never);
}

// Issues the TMA load of the Q tile of unit u into the staging buffer.
template <int D, int BN>
__device__ __forceinline__ void load_q(const CUtensorMap* mapQ, const AttnParams& p, int u, uint8_t* q_stage,
                                       uint64_t* bar) {
  using C = AttnCfg<D, BN>;
  int b, h, qt;
  decode_unit(p, u, b, h, qt);
  mbar_arrive_expect_tx(bar, C::kQBytes);
  for (int i = 0; i < C::kBoxes; ++i)
    tma_load_3d(q_stage + i * 128 * 128, mapQ, bar, 64 * i, qt * 128, b * p.n_heads + h);
}

// First unit at or after u (stepping by stride) that has at least one tile.
template <int BN, int MODE>
__device__ __forceinline__ int next_nonempty_unit(const AttnParams& p, int u, int stride) {
  for (; u < p.n_units; u += stride) {
    if (MODE != kSparse) return u;
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    auto it = make_iter<BN, MODE>(p, b, h / p.group, qt);
    int kb, bits;
    if (it.next(kb, bits)) return u;
  }
  return INT_MAX;
}

// Loads this thread's kCols columns of an S tile (one or two 32-column
// loads, one wait) and applies the causal / support masks.
template <int kCols>
__device__ __forceinline__ void load_s_half(uint32_t addr, float (&s)[kCols], bool attend, int lim) {
  uint32_t va[32], vb[32];
  tmem_ld_32x32b_x32(addr, va);
  if constexpr (kCols == 64) {
    tmem_ld_32x32b_x32(addr + 32, vb);
    tmem_ld_wait(va, vb);
  } else {
    tmem_ld_wait(va);
  }
#pragma unroll
  for (int e = 0; e < 32; ++e) s[e] = __uint_as_float(va[e]);
  if constexpr (kCols == 64) {
#pragma unroll
    for (int e = 0; e < 32; ++e) s[32 + e] = __uint_as_float(vb[e]);
  }
  if (!attend) {
#pragma unroll
    for (int c = 0; c < kCols; ++c) s[c] = -INFINITY;
  } else if (lim < kCols - 1) {
    // keys with column c > lim are in the future of this row
#pragma unroll
    for (int c = 0; c < kCols; ++c) s[c] = (c > lim) ? -INFINITY : s[c];
  }
}

// Exchange of one float per row between the two softmax halves: thread
// (half, row) publishes v and gets its partner's value.  Double-buffered by
// phase; bounded wait.
template <class SB>
__device__ __forceinline__ void half_publish(SB& sb, int phase, int half, int row, int lane, float v) {
  sb.xbuf[phase & 1][half][row] = v;
  __syncwarp();
  if (lane == 0) mbar_arrive(&sb.xch);
}

template <class SB>
__device__ __forceinline__ bool half_collect(SB& sb, int& phase, int half, int row, float& other,
                                             volatile int* abort) {
  if (!warp_wait(&sb.xch, phase & 1, abort)) return false;
  other = sb.xbuf[phase & 1][half ^ 1][row];
  ++phase;
  return true;
}

template <class SB>
__device__ __forceinline__ bool half_exchange(SB& sb, int& phase, int half, int row, int lane,
                                              float v, float& other, volatile int* abort) {
  half_publish(sb, phase, half, row, lane, v);
  return half_collect(sb, phase, half, row, other, abort);
}

// ------------------------------------------------------------------- softmax
// Warpgroup `half` of the softmax owns, for every query row of the tile,
// key columns [half*BN/2, (half+1)*BN/2) of S and output columns
// [half*D/2, (half+1)*D/2) of O.
template <int D, int BN, int MODE>
__device__ void attn_softmax(const CUtensorMap* mapQ, const AttnParams& p, int half, uint32_t tmem,
                             uint8_t* q_stage, SharedBarriers<AttnCfg<D, BN>::kRingK, AttnCfg<D, BN>::kRingV>& sb) {
  using C = AttnCfg<D, BN>;
  constexpr int kCols = BN / 2;  // S columns per half
  constexpr int kOCols = D / 2;  // O columns per half
  // Pairs of every 8 whose exponential runs on the FMA pipe; the block-mass
  // variant keeps the hardware ex2 throughout for its sums.
  constexpr int kEmu = (MODE == kDenseMass) ? 0 : WISE_EMU_PAIRS;
  volatile int* abort = &sb.abort;
  const int r = threadIdx.x & 127;  // query row within the tile
  const int wq = r >> 5, lane = r & 31;
  const bool leader = (half == 0 && r == 0);
  const uint32_t lane_tmem = tmem + ((uint32_t)(wq * 32) << 16);
  constexpr float kRescaleThreshold = 8.0f;  // log2 units: P stays <= 256
  const int G = gridDim.x;
  // Per-CTA scratch: [n_blocks][2][128] log2 partial masses, then
  // [2][4][n_blocks] per-warp column sums.
  float* scratch = p.scratch + (size_t)blockIdx.x * p.n_blocks * 264;
  float* warp_sums = scratch + (size_t)p.n_blocks * 256;

  // Q pipeline: the staging buffer holds the Q of unit q_next; copy_next()
  // moves it into TMEM buffer n_q & 1 and prefetches the following one.
  int q_next = next_nonempty_unit<BN, MODE>(p, blockIdx.x, G);
  int n_q = 0, x_phase = 0, j = 0;
  if (leader && q_next != INT_MAX) load_q<D, BN>(mapQ, p, q_next, q_stage, &sb.q_full);
  bool ok = true;
  auto copy_next = [&]() -> bool {
    if (!warp_wait(&sb.q_full, n_q & 1, abort)) return false;
    const uint32_t q_col = C::kTmemQ + (n_q & 1) * C::kTmemQCols;
    if (half < C::kBoxes) {
      const uint32_t box = smem_u32(q_stage + half * 128 * 128) + r * 128;
      uint32_t w[32];
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const uint4 v = ld_shared_v4(box + ((c ^ (r & 7)) << 4));
        w[4 * c + 0] = v.x;
        w[4 * c + 1] = v.y;
        w[4 * c + 2] = v.z;
        w[4 * c + 3] = v.w;
      }
      tmem_st_32x32b_x32(lane_tmem + q_col + half * 32, w);
      tmem_st_wait();
    }
    tc_fence_before_sync();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.q_tmem[n_q & 1]);
    const int following = next_nonempty_unit<BN, MODE>(p, q_next + G, G);
    if (leader && following != INT_MAX) {
      // Every warp has read the staging buffer once q_tmem completes.
      if (!mbar_wait(&sb.q_tmem[n_q & 1], (n_q >> 1) & 1, abort)) return false;
      load_q<D, BN>(mapQ, p, following, q_stage, &sb.q_full);
    }
    q_next = following;
    ++n_q;
    return true;
  };
  if (q_next != INT_MAX && !copy_next()) ok = false;

  for (int u = blockIdx.x; u < p.n_units && ok; u += G) {
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    auto it = make_iter<BN, MODE>(p, b, h / p.group, qt);
    const int row = qt * 128 + r;
    const int half_bit = (BN == 64) ? (1 << (r >> 6)) : 1;
    float m_ref = -INFINITY, l = 0.0f;
    int jj = 0, kb, bits, last_kb = -1;
    bool have = it.next(kb, bits);
    // The next unit's Q goes into the other TMEM buffer while this one runs.
    if (have && q_next != INT_MAX && !copy_next()) {
      ok = false;
      break;
    }
    while (have) {
      int nkb, nbits;
      const bool more = it.next(nkb, nbits);
      last_kb = kb;
      const uint32_t s_col = C::kTmemS + (j & 1) * C::kTmemSCols;
      if (!warp_wait(&sb.s_full[j & 1], (j >> 1) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const int k0 = kb * BN + half * kCols;
      const bool attend = (bits & half_bit) != 0;
      const int lim = row - k0;  // keys k0 + c with c > lim are in the future
      const uint32_t s_addr = lane_tmem + s_col + half * kCols;
      float s[kCols];
      load_s_half<kCols>(s_addr, s, attend, lim);
      const float mx_local = row_max(s);
      // The partner half's maximum is needed before the exponentials can be
      // trusted; publish now and collect after them.  Past a unit's first
      // tile the running max rarely moves, so the exponentials are computed
      // speculatively against it and redone only where it did move.
      half_publish(sb, x_phase, half, r, lane, mx_local);
      const bool first_tile = (jj == 0);
      const float m_old = m_ref;
      float rowsum = 0.0f;
      const bool masked = !attend || lim < kCols - 1;
      if (!first_tile) rowsum = exp2_scaled<kEmu>(s, p.scale_log2, m_old == -INFINITY ? 0.0f : m_old, masked);
      float mx_other;
      if (!half_collect(sb, x_phase, half, r, mx_other, abort)) {
        ok = false;
        break;
      }
      const float m_tile = fmaxf(mx_local, mx_other) * p.scale_log2;
      float alpha = 1.0f;
      bool rescale = false;
      if (m_tile > m_ref + kRescaleThreshold) {
        alpha = ex2_approx(m_ref - m_tile);
        rescale = (m_ref != -INFINITY);
        m_ref = m_tile;
        l *= alpha;
      }
      const float m_use = (m_ref == -INFINITY) ? 0.0f : m_ref;
      if (first_tile) {
        rowsum = exp2_scaled<kEmu>(s, p.scale_log2, m_use, masked);
      } else if (__any_sync(0xffffffffu, m_ref != m_old)) {
        // Redo the rows whose running max moved (S is still in TMEM).
        float t[kCols];
        load_s_half<kCols>(s_addr, t, attend, lim);
        const float tsum = exp2_scaled<kEmu>(t, p.scale_log2, m_use, masked);
        if (m_ref != m_old) {
          rowsum = tsum;
#pragma unroll
          for (int c = 0; c < kCols; ++c) s[c] = t[c];
        }
      }
      // P as bf16 pairs: keys [half*kCols, (half+1)*kCols) of the row go to
      // columns [half*kCols/2, (half+1)*kCols/2) of this tile's S buffer.
      // The stores complete while the bookkeeping below runs.
#pragma unroll
      for (int c = 0; c < kCols / 32; ++c) {
        uint32_t w[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) w[e] = pack_bf16x2(s[32 * c + 2 * e], s[32 * c + 2 * e + 1]);
        tmem_st_32x32b_x16(lane_tmem + s_col + half * (kCols / 2) + 16 * c, w);
      }
      l += rowsum;  // this half's part of the row sum
      if (MODE == kDenseMass)
        scratch[((size_t)kb * 2 + half) * 128 + r] = rowsum > 0.0f ? m_ref + lg2_approx(rowsum) : -INFINITY;
      // O is rescaled only after the previous P V completed.  tcgen05.ld/st
      // are warp-collective: the warp rescales together, lanes whose max did
      // not move use a factor of 1.
      if (jj > 0 && __any_sync(0xffffffffu, rescale)) {
        if (!warp_wait(&sb.o_full, (j - 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const float f = rescale ? alpha : 1.0f;
        const uint32_t o_col = C::kTmemO + half * kOCols;
#pragma unroll
        for (int c = 0; c < kOCols / 16; ++c) {
          uint32_t v[16];
          tmem_ld_32x32b_x16(lane_tmem + o_col + 16 * c, v);
          tmem_ld_wait(v);
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * f);
          tmem_st_32x32b_x16(lane_tmem + o_col + 16 * c, v);
        }
      }
      tmem_st_wait();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sb.p_full[j & 1]);
      ++j;
      ++jj;
      kb = nkb;
      bits = nbits;
      have = more;
    }
    if (!ok) break;
    // ---- epilogue: O / l over both halves
    float l_other = 0.0f;
    if (!half_exchange(sb, x_phase, half, r, lane, l, l_other, abort)) {
      ok = false;
      break;
    }
    const float l_row = half == 0 ? l + l_other : l_other + l;  // same order in both halves
    if (jj > 0) {
      if (!warp_wait(&sb.o_full, (j - 1) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
    }
    const float inv_l = l_row > 0.0f ? 1.0f / l_row : 0.0f;
    __nv_bfloat16* orow = p.O + ((size_t)(b * p.n_heads + h) * p.seqlen + row) * D + half * kOCols;
#pragma unroll
    for (int c = 0; c < kOCols / 16; ++c) {
      uint32_t v[16];
      if (jj > 0) {
        tmem_ld_32x32b_x16(lane_tmem + C::kTmemO + half * kOCols + 16 * c, v);
        tmem_ld_wait(v);
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = 0u;
      }
      uint32_t w[8];
#pragma unroll
      for (int e = 0; e < 8; ++e)
        w[e] = pack_bf16x2(__uint_as_float(v[2 * e]) * inv_l, __uint_as_float(v[2 * e + 1]) * inv_l);
      if (row < p.seqlen) {
        uint4* dst = reinterpret_cast<uint4*>(orow + 16 * c);
        dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
        dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
      }
    }
    // ---- epilogue: block mass (Eq. 5)
    if (MODE == kDenseMass) {
      const float lse = m_ref + lg2_approx(l_row);
      const int n_kt = last_kb + 1;
      for (int t = 0; t < n_kt; ++t) {
        const float lc = scratch[((size_t)t * 2 + half) * 128 + r];
        float v = (row < p.seqlen) ? ex2_approx(lc - lse) : 0.0f;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if (lane == 0) warp_sums[(half * 4 + wq) * p.n_blocks + t] = v;
      }
      // The exchange barrier orders the eight warps' global writes before
      // the reads below (release/acquire at CTA scope).
      float unused;
      if (!half_exchange(sb, x_phase, half, r, lane, 0.0f, unused, abort)) {
        ok = false;
        break;
      }
      constexpr int kHalves = 128 / BN;  // query blocks per tile
      const float inv_b = 1.0f / (float)BN;
      const int tid = half * 128 + r;
      for (int e = tid; e < kHalves * p.n_blocks; e += 256) {
        const int hf = e / p.n_blocks, t = e % p.n_blocks;
        const int qblock = qt * kHalves + hf;
        if (qblock >= p.n_blocks) continue;
        float* out = p.blockmass + ((size_t)(b * p.n_heads + h) * p.n_blocks + qblock) * p.n_blocks + t;
        if (t < n_kt) {
          float sum = 0.0f;
          if (BN == 128) {
#pragma unroll
            for (int w = 0; w < 8; ++w) sum += warp_sums[w * p.n_blocks + t];
          } else {
#pragma unroll
            for (int hh = 0; hh < 2; ++hh)
#pragma unroll
              for (int w = 2 * hf; w < 2 * hf + 2; ++w) sum += warp_sums[(hh * 4 + w) * p.n_blocks + t];
          }
          sum *= inv_b;
          *out = (p.step == 0) ? sum : *out + sum;
        } else if (p.step == 0) {
          *out = 0.0f;
        }
      }
      // warp_sums is rewritten by the next unit.
      if (!half_exchange(sb, x_phase, half, r, lane, 0.0f, unused, abort)) {
        ok = false;
        break;
      }
    }
  }
  if (!ok) {
    raise_status(p, &sb.abort, kStatusTimeout);
    if (leader && n_q > 0) {
      // Let a Q copy still in flight land before shared memory is released.
      int never = 0;
      mbar_wait(&sb.q_full, n_q & 1, &never);
    }
  }
}

// -------------------------------------------------------------------- kernel
template <int D, int BN, int MODE>
__global__ void __launch_bounds__(AttnCfg<D, BN>::kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                const __grid_constant__ CUtensorMap mapV, const AttnParams p) {
  using C = AttnCfg<D, BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_stage = smem;             // one Q tile
  uint8_t* ring = smem + C::kQBytes;   // kRing K/V entries
  __shared__ SharedBarriers<C::kRingK, C::kRingV> sb;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    sb.abort = 0;
    for (int i = 0; i < C::kRingK; ++i) {
      mbar_init(&sb.k_full[i], 1);
      mbar_init(&sb.k_empty[i], 1);
    }
    for (int i = 0; i < C::kRingV; ++i) {
      mbar_init(&sb.v_full[i], 1);
      mbar_init(&sb.v_empty[i], 1);
    }
    mbar_init(&sb.q_full, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sb.q_tmem[b], 8);
      mbar_init(&sb.s_full[b], 1);
      mbar_init(&sb.buf_free[b], 1);
      mbar_init(&sb.p_full[b], 8);
    }
    mbar_init(&sb.o_full, 1);
    mbar_init(&sb.xch, 8);
    mbar_init(&sb.s_done, 1);
    mbar_init(&sb.pv_done, 1);
    fence_mbar_init();
  }
  if (warp == C::kProducerWarp && lane == 0) {
    tma_prefetch_map(&mapQ);
    tma_prefetch_map(&mapK);
    tma_prefetch_map(&mapV);
  }
  if (warp == C::kMmaSWarp) {
    tmem_alloc(&sb.tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sb.tmem_base;

  if (warp < 8) {
    attn_softmax<D, BN, MODE>(&mapQ, p, warp >> 2, tmem, q_stage, sb);
  } else if (warp == C::kProducerWarp) {
    if (lane == 0) attn_producer<D, BN, MODE>(&mapK, &mapV, p, ring, sb);
  } else if (warp == C::kMmaSWarp) {
    if (lane == 0) attn_mma_s<D, BN, MODE>(p, tmem, ring, sb);
  } else if (warp == C::kMmaPVWarp) {
    if (lane == 0) attn_mma_pv<D, BN, MODE>(p, tmem, ring, sb);
  }

  __syncwarp();
  tc_fence_before_sync();
  __syncthreads();
  if (warp == C::kMmaSWarp) {
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
