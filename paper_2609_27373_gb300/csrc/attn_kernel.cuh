// Causal flash attention on tcgen05 tensor cores, in three variants:
//   kDense      O = softmax(Q K^T * scale + M) V                  (Eq. 2)
//   kDenseMass  the same, plus the block attention mass of the step (Eq. 5)
//               accumulated into blockmass
//   kSparse     key blocks restricted to the selected support      (Eqs. 7-8)
//
// Work decomposition.  A unit is one 128-row query tile of one (batch, head);
// units are numbered in order of decreasing causal length.  The persistent
// grid (one CTA per SM) deals them out in a snake order (CTA c takes unit
// k*G + c in even rounds k and k*G + G-1-c in odd rounds), which evens out
// the per-CTA sums of the decreasing lengths.  Each unit walks its list of
// key tiles (128 keys each): every tile of the causal prefix (dense), or the
// tiles holding blocks of the support (sparse).  With a block B of 32 or 64 a
// query tile covers S = 128 / B query blocks and a key tile S key blocks; the
// unit walks the union of its query blocks' lists, and each tile carries an
// S x S mask of the (query block, key block) pairs that attend.
//
// Both products run with the A operand in tensor memory: Q is copied into
// TMEM once per unit, so that its staging buffer can already receive the next
// unit's Q.  (With two threads issuing, MMAs with A in shared memory run at
// the same rate; one thread alone issues at most about one MMA per 89 clk
// against the 64 clk an M128/N128/K16 step takes, hence two issuers.)
//   S = Q K^T    Q copied per unit from shared memory into TMEM with
//                tcgen05.cp (ordered before the MMAs that read it), K from
//                shared memory (K-major);
//   O += P V     P written by the softmax into TMEM, V from shared memory
//                (MN-major).
// TMEM (512 columns, 448 used): Q (64 columns), one S buffer (128 columns), P
// double-buffered across tiles (2 x 64 columns), O (128 columns).  S(j+1) is
// issued as soon as the softmax has read S(j) into registers, so the S product
// never waits for a P V, and P(j) waits only for P V(j-2).  (With two S
// buffers and one P buffer instead, P(j) has to wait for P V(j-1), which may
// sit behind an S product in the tensor pipe: a serial P -> P V -> P chain
// that measured slower.)  The Q of the next unit is copied in once the last S
// product of the current unit has completed.
//
// Warp roles (384 threads; warp 11 only completes warpgroup 2):
//   warp 8     producer.  Walks the CTA's units, validates the support lists,
//              and publishes the tile schedule in three shared-memory rings:
//              ring w (w = 0, 1) holds the tiles j with j & 1 == w for softmax
//              warpgroup w (ring 0 also the units without tiles), ring 2 every
//              tile for the two MMA threads, and each ring ends with an end
//              marker; issues the
//              TMA loads of Q (staging buffer), K (ring of kRingK) and V (ring
//              of kRingV) in the order Q, K(0), K(1), V(0), K(2), V(1), ...
//   warp 9     S issuer: copies each unit's Q into TMEM and issues
//              S(j) = Q K(j)^T once S(j-1) has been read.
//   warp 10    P V issuer: O += P(j) V(j) once the softmax has written P(j).
//              A tcgen05.mma issue blocks its thread while the tensor core
//              drains earlier instructions, so the two products are issued
//              from two threads.
//   warps 0-3 and 4-7  softmax warpgroups 0 and 1.  Warpgroup w handles the
//              tiles j with j & 1 == w (so it always writes P buffer w); thread
//              t of a warpgroup owns query row t (= TMEM lane t) and the whole
//              row of each of its tiles.  The online softmax runs in the log2
//              domain with one running max m per row shared by both
//              warpgroups: for tile j, the handler needs m after tile j-1
//              (from the other warpgroup, through shared memory) and
//              publishes m after tile j; O is rescaled only when m grows by
//              more than 2^8.  Each warpgroup keeps its own part of the row
//              sum; the two parts are combined at the end of the unit.  Since
//              the two warpgroups work on different tiles, one computes
//              exponentials while the other loads S or writes P.
//   Epilogue.  The warpgroup that handled the unit's last tile (L) writes
//              O / l to global memory (and, for kDenseMass, the block
//              masses); the other one (E) only publishes its part of the row
//              sum and goes on with the next unit's first tile, which is
//              always its own.  The first P V of a unit waits until L has
//              read O.
//
// Every wait is bounded (kWaitLimitNs); a wait that runs out sets the status
// word and an abort flag, and every role unwinds.
#pragma once

#include <cuda_bf16.h>
#include <limits.h>
#include <stdint.h>

#include "attn_common.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace wise {

template <int D>
struct AttnCfg {
  static constexpr int kBoxes = (D + 63) / 64;          // 64-column TMA boxes per row tile
  static constexpr int kQBytes = kBoxes * 128 * 128;    // one 128-row Q tile (staging)
  static constexpr int kKVBytes = kBoxes * kTileN * 128; // one 128-row K or V tile (one ring entry)
  // Static shared memory (barriers, schedule ring, row exchange buffers).
  static constexpr int kStaticReserve = 10 * 1024;
  // Dynamic shared memory available after the 1024-byte alignment slack.
  static constexpr int kBudget = 227 * 1024 - 1024 - kStaticReserve;
  // Epilogue staging: per softmax warp of L, 32 rows x 64 columns of O
  // (one 128-byte-swizzled TMA box).
  static constexpr int kOutBytes = 4 * 32 * 128;
  // Block-mass epilogue: per-warp column sums [2 buffers][4 warps][key
  // blocks] for up to kMassWsBlocks key blocks (more go to the global scratch).
  static constexpr int kMassWsBlocks = 128;
  static constexpr int kMassWsBytes = 2 * 4 * kMassWsBlocks * 4;
  static constexpr int kRingFit = (kBudget - kQBytes - kOutBytes - kMassWsBytes) / kKVBytes;
  static constexpr int kRing = kRingFit > 12 ? 12 : kRingFit;
  static constexpr int kRingK = (kRing + 1) / 2;  // K tiles (consumed by S)
  static constexpr int kRingV = kRing / 2;        // V tiles (consumed by P V)
  static constexpr int kSmemBytes = kQBytes + kRing * kKVBytes + kOutBytes + kMassWsBytes + 1024;
  // At least 116 KB so that a single CTA resides per SM (it owns all 512
  // TMEM columns).
  static constexpr int kSmemLaunch = kSmemBytes > 116 * 1024 ? kSmemBytes : 116 * 1024;
  static constexpr uint32_t kTmemQ = 0;       // Q: 128 bf16 per row
  static constexpr uint32_t kTmemS = 128;     // one S buffer
  static constexpr uint32_t kTmemP = 256;     // two P buffers of 64 columns
  static constexpr uint32_t kTmemPCols = 64;
  static constexpr uint32_t kTmemO = 384;     // O accumulator
  static constexpr uint32_t kTmemCols = 512;
  // Warps 0-7 softmax, 8 producer, 9 and 10 MMA issuers, 11 schedule
  // stager (sparse with blocks of 32 or 64; otherwise idle, it completes
  // warpgroup 2 for setmaxnreg).  Launch: 384 x 168 registers;
  // after the split 256 x kRegsSoftmax + 128 x kRegsOther = 64512.
  static constexpr int kThreads = 384;
  static constexpr int kRegsSoftmax = 216;
  static constexpr int kRegsOther = 72;
  static constexpr int kProducerWarp = 8;
  static constexpr int kMmaSWarp = 9;   // issues S = Q K^T, owns the TMEM allocation
  static constexpr int kMmaPVWarp = 10; // issues O += P V
  static_assert(kRingV >= 1 && kRingK >= 2, "shared memory budget");
  static_assert(D <= 128, "TMEM budget");
  static_assert(256 * kRegsSoftmax + 128 * kRegsOther <= kThreads * 168, "register split");
};

// Sparse tile schedules staged by warp 11 (blocks of 32 and 64, S > 1 lists
// per unit): entries per slot (a unit's tiles, as schedule keys), the key
// tiles a staged unit may span, and the slots.  A launch stages when every
// unit fits: cap * S <= kStageKeys (each accepted list entry adds at most one
// tile) and n_qtiles <= kStageTiles.  With one list per unit (block 128) the
// producer's own merge measured faster than staging (4K late step 68.5
// against 74 us).
constexpr int kStageKeys = 128;
constexpr int kStageTiles = 256;
constexpr int kStageSlots = 4;
template <int BLK, int MODE>
__device__ __forceinline__ bool sched_staging(const AttnParams& p) {
  constexpr int S = kTileN / BLK;
  return MODE == kSparse && S > 1 && p.cap <= kStageKeys / S && p.n_qtiles <= kStageTiles;
}

template <int RK, int RV>
struct SharedState {
  uint64_t k_full[RK], k_empty[RK], v_full[RV], v_empty[RV];
  uint64_t sched_full[3][kSchedSlots], sched_empty[3][kSchedSlots];
  // A parity wait is exact only while the barrier is at most one phase away
  // from the awaited one.  Barriers whose waiters may arrive late (after the
  // next phase could complete) or early (before the previous phase has
  // completed) therefore exist once per buffer: a second completion of the
  // same barrier needs work that the waiter itself has not released yet, and
  // its previous completion is implied by work the waiter has already seen.
  uint64_t q_full;        // Q tile landed in the staging buffer (TMA)
  uint64_t q_stage_free;  // staging buffer copied into TMEM (S thread commit)
  uint64_t q_free;        // last S of a unit completed (S thread commit)
  uint64_t s_full[2];     // S(j) written, j & 1 == b (S thread commit)
  uint64_t s_free[2];     // S(j) read by its softmax warpgroup, j & 1 == b (4 warps)
  uint64_t p_full[2];     // P(j) written, j & 1 == b (4 warps of warpgroup b)
  uint64_t o_full[2];     // P V(j) completed, j & 1 == b (P V thread commit); frees P buffer b
  uint64_t o_free;        // the epilogue read O (4 warps of L)
  uint64_t m_pub[2][2];   // warpgroup w published its running max, slot = its tile count & 1
  uint64_t l_pub[2];      // warpgroup w, as E, published its row-sum part of a unit
  uint64_t l_ack[2];      // the other warpgroup (L) read that part
  uint64_t epi[2];        // the 4 warps of warpgroup w wrote their block-mass sums
  uint64_t s_done, pv_done;
  int4 sched[3][kSchedSlots];
  float mx[2][2][128];   // [warpgroup][slot][row] running max after a tile
  float lx[2][128];      // [warpgroup][row] E's row-sum part at the end of a unit
  float lm[2][128];      // [warpgroup][row] the max that part refers to
  // Staged tile schedules (slot = the unit's position in the CTA's sequence
  // mod kStageSlots): the keys of the unit's tiles and their number n (-1 - n when a
  // count or a list entry of the unit was invalid).
  uint64_t list_full[kStageSlots];   // staged (warp 11)
  uint64_t list_empty[kStageSlots];  // the producer has read the slot
  int32_t stage_keys[kStageSlots][kStageKeys];
  int32_t stage_n[kStageSlots];
  uint32_t stage_tmask[kStageTiles];  // warp 11 scratch: mask of each key tile
  uint32_t tmem_base;
  int abort;
};

// -------------------------------------------------------- schedule stager
// Sparse launches that stage (sched_staging): warp 11 walks the CTA's units
// in the producer's order, at most kStageSlots units ahead, and turns each unit's S
// support lists into its tile schedule in shared memory, with the 32 lanes
// working together: an entry of list q is accepted if it lies in [0, q0 + q]
// and exceeds every accepted entry before it in its list (= every in-range
// entry before it: an in-range entry that was not accepted lies below an
// accepted one), which a prefix max over the list finds; the accepted key
// blocks are OR-ed into a mask per key tile; the tiles with a non-empty mask
// are compacted in ascending order.  The producer then reads a unit's keys
// from shared memory instead of merging the lists itself, one dependent
// global load per list entry on a thread that shares its scheduler with two
// busy softmax warps.
template <int D, int BLK, int MODE>
__device__ void attn_sched_stager(const AttnParams& p, SharedState<AttnCfg<D>::kRingK, AttnCfg<D>::kRingV>& sb) {
  constexpr int S = kTileN / BLK;
  constexpr int kCap = kStageKeys / S;      // list positions staged per query block (>= cap)
  constexpr int kRegs = kStageKeys / 32;    // entry e = lane + 32 i in register i
  constexpr int kRegsPerList = kCap / 32;   // list q: registers q * kRegsPerList ..
  const int lane = threadIdx.x & 31;
  volatile int* abort = &sb.abort;
  const int G = gridDim.x, c = blockIdx.x;
  int n_st = 0;
  bool ok = true;
  for (int k = 0; ok && k * G < p.n_units; ++k) {
    const int u = k * G + ((k & 1) ? G - 1 - c : c);
    if (u >= p.n_units) continue;
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    const int q0 = qt * S;
    const size_t row0 = ((size_t)b * p.n_kv_heads + h / p.group) * p.n_blocks + q0;
    const int slot = n_st % kStageSlots;
    // The producer has read the schedule that used the slot before.
    if (n_st >= kStageSlots && !warp_wait(&sb.list_empty[slot], ((n_st / kStageSlots) - 1) & 1, abort, p.wait_ns)) {
      ok = false;
      break;
    }
    int bad = 0;
    int cnt[S];
#pragma unroll
    for (int q = 0; q < S; ++q) cnt[q] = (q0 + q < p.n_blocks) ? __ldg(p.counts + row0 + q) : 0;
    // The entries are loaded alongside the counts (every position below cap
    // exists), so that the unit costs one memory latency.
    int v[kRegs];
    bool live[kRegs], acc[kRegs];
#pragma unroll
    for (int i = 0; i < kRegs; ++i) {
      const int q = i / kRegsPerList, x = (i % kRegsPerList) * 32 + lane;
      v[i] = (q0 + q < p.n_blocks && x < p.cap) ? __ldg(p.idx + (row0 + q) * p.cap + x) : -1;
    }
#pragma unroll
    for (int q = 0; q < S; ++q) cnt[q] = (q0 + q < p.n_blocks) ? clamp_count(cnt[q], p.cap, bad) : 0;
#pragma unroll
    for (int i = 0; i < kRegs; ++i) live[i] = (i % kRegsPerList) * 32 + lane < cnt[i / kRegsPerList];
    int carry = -1;  // max of the in-range entries of the list's earlier registers
#pragma unroll
    for (int i = 0; i < kRegs; ++i) {
      const int q = i / kRegsPerList;
      if (i % kRegsPerList == 0) carry = -1;
      const bool in_range = live[i] && v[i] >= 0 && v[i] <= q0 + q;
      int m = in_range ? v[i] : -1;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, m, o);
        if (lane >= o) m = max(m, t);
      }
      int before = __shfl_up_sync(0xffffffffu, m, 1);
      before = max(lane == 0 ? -1 : before, carry);
      acc[i] = in_range && v[i] > before;
      if (live[i] && !acc[i]) bad = 1;
      carry = max(carry, __shfl_sync(0xffffffffu, m, 31));
    }
    // Masks of the key tiles 0..qt (every accepted block lies in one).
    for (int t = lane; t <= qt; t += 32) sb.stage_tmask[t] = 0u;
    __syncwarp();
#pragma unroll
    for (int i = 0; i < kRegs; ++i)
      if (acc[i]) atomicOr(&sb.stage_tmask[v[i] / S], 1u << ((i / kRegsPerList) * S + v[i] % S));
    __syncwarp();
    int n = 0;
    for (int t0 = 0; t0 <= qt; t0 += 32) {
      const int t = t0 + lane;
      const uint32_t m = t <= qt ? sb.stage_tmask[t] : 0u;
      const uint32_t bal = __ballot_sync(0xffffffffu, m != 0u);
      if (m) sb.stage_keys[slot][n + __popc(bal & ((1u << lane) - 1u))] = (int)((uint32_t)t | (m << 16));
      n += __popc(bal);
    }
    bad = __any_sync(0xffffffffu, bad);
    if (lane == 0) sb.stage_n[slot] = bad ? -1 - n : n;
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.list_full[slot]);
    ++n_st;
  }
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
}

// ------------------------------------------------------------------ producer
template <int D, int BLK, int MODE>
__device__ void attn_producer(const CUtensorMap* mapQ, const CUtensorMap* mapK, const CUtensorMap* mapV,
                              const AttnParams& p, uint8_t* q_stage, uint8_t* ring,
                              SharedState<AttnCfg<D>::kRingK, AttnCfg<D>::kRingV>& sb) {
  using C = AttnCfg<D>;
  constexpr int RK = C::kRingK, RV = C::kRingV;
  uint8_t* k_ring = ring;
  uint8_t* v_ring = ring + RK * C::kKVBytes;
  volatile int* abort = &sb.abort;
  int jk = 0, jv = 0, nq = 0, bad = 0;
  int jt = 0, n_empty = 0;  // tiles and units without tiles scheduled so far
  int n_units = 0;          // units walked so far
  const bool staged = sched_staging<BLK, MODE>(p);
  bool ok = true;
  // Writes the next entry of a ring.  Its position follows from the counts:
  // the MMA ring holds every tile, ring 1 the odd tiles, ring 0 the even
  // tiles and the units without tiles.
  auto emit = [&](int ring_w, int kb, int u, int flags, int t) -> bool {
    const int e = ring_w == kMmaRing ? jt : ring_w == 1 ? (jt >> 1) : ((jt + 1) >> 1) + n_empty;
    const int slot = e % kSchedSlots;
    if (e >= kSchedSlots &&
        !mbar_wait(&sb.sched_empty[ring_w][slot], ((e / kSchedSlots) - 1) & 1, abort, p.wait_ns))
      return false;
    sb.sched[ring_w][slot] = make_int4(kb, u, flags, t);
    mbar_arrive(&sb.sched_full[ring_w][slot]);  // release: the entry is visible to whoever acquires the phase
    return true;
  };
  auto load = [&](const CUtensorMap* map, uint8_t* base, uint64_t* full, uint64_t* empty, int R, int& j, int kb,
                  int z) -> bool {
    const int slot = j % R;
    if (j >= R && !mbar_wait(&empty[slot], ((j / R) - 1) & 1, abort, p.wait_ns)) return false;
    mbar_arrive_expect_tx(&full[slot], C::kKVBytes);
    for (int i = 0; i < C::kBoxes; ++i)
      tma_load_3d(base + slot * C::kKVBytes + i * kTileN * 128, map, &full[slot], 64 * i, kb * kTileN, z);
    ++j;
    return true;
  };
  const int G = gridDim.x, c = blockIdx.x;
  int prev_kb = 0, prev_z = 0;
  bool have_prev = false;
  for (int k = 0; ok && k * G < p.n_units; ++k) {
    const int u = k * G + ((k & 1) ? G - 1 - c : c);
    if (u >= p.n_units) continue;  // only in the last, partial round
    int b, h, qt;
    decode_unit(p, u, b, h, qt);
    const int kvh = h / p.group;
    const int z = b * p.n_kv_heads + kvh;
    // The unit's tiles: from warp 11's staged schedule, or merged here.
    const int lslot = n_units % kStageSlots;
    int st_n = 0, st_t = 0;
    TileIter<BLK, MODE> it;
    if (staged) {
      if (!mbar_wait(&sb.list_full[lslot], (n_units / kStageSlots) & 1, abort, p.wait_ns)) {
        ok = false;
        break;
      }
      st_n = sb.stage_n[lslot];
      if (st_n < 0) {
        bad = 1;
        st_n = -1 - st_n;
      }
    } else {
      it = make_iter<BLK, MODE>(p, b, kvh, qt);
    }
    auto next_tile = [&](int& kt, uint32_t& m) -> bool {
      if (staged) {
        if (st_t >= st_n) return false;
        const int key = sb.stage_keys[lslot][st_t++];
        kt = key & 0xFFFF;
        m = (uint32_t)key >> 16;
        return true;
      }
      return it.next(kt, m);
    };
    int kb;
    uint32_t mask;
    bool have = next_tile(kb, mask);
    if (!have) {
      if (!emit(0, 0, u, kEntEmpty, 0)) ok = false;
      ++n_empty;
    }
    bool first = true;
    const int unit_ix = nq;  // index of this unit among the units with tiles
    for (int t = 0; have && ok; ++t) {
      int nkb;
      uint32_t nmask;
      const bool more = next_tile(nkb, nmask);
      const int flags = (first ? kEntFirst : 0) | (more ? 0 : kEntLast) | (unit_ix << kEntUnitShift);
      const int key = (int)((uint32_t)kb | (mask << 16));
      if (!emit(kMmaRing, key, u, flags, t) || !emit(jt & 1, key, u, flags, t)) {
        ok = false;
        break;
      }
      ++jt;
      if (first) {
        // The first copy: the previous kernel of the stream has completed.
        if (nq == 0) griddep_wait();
        // The staging buffer is free once the previous unit's Q is in TMEM.
        if (nq >= 1 && !mbar_wait(&sb.q_stage_free, (nq - 1) & 1, abort, p.wait_ns)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&sb.q_full, C::kQBytes);
        for (int i = 0; i < C::kBoxes; ++i)
          tma_load_3d(q_stage + i * 128 * 128, mapQ, &sb.q_full, 64 * i, qt * 128, b * p.n_heads + h);
        ++nq;
      }
      if (!load(mapK, k_ring, sb.k_full, sb.k_empty, RK, jk, kb, z)) {
        ok = false;
        break;
      }
      if (have_prev && !load(mapV, v_ring, sb.v_full, sb.v_empty, RV, jv, prev_kb, prev_z)) {
        ok = false;
        break;
      }
      prev_kb = kb;
      prev_z = z;
      have_prev = true;
      kb = nkb;
      mask = nmask;
      have = more;
      first = false;
    }
    if (staged) {
      mbar_arrive(&sb.list_empty[lslot]);  // the schedule has been read
    } else {
      bad |= it.bad;
    }
    ++n_units;
  }
  if (ok && have_prev && !load(mapV, v_ring, sb.v_full, sb.v_empty, RV, jv, prev_kb, prev_z)) ok = false;
  for (int rw = 0; rw < 3 && ok; ++rw)
    if (!emit(rw, 0, 0, kEntEnd, jt)) ok = false;
  // The MMA threads read tile j's entry of the MMA ring once K(j) (S thread)
  // or V(j) (P V thread) has landed, the entry being written before either
  // is loaded.  The end marker is announced the same way: the next K and V
  // barriers complete without a copy, once their slots' last loads have been
  // consumed.
  if (ok && jk >= RK && !mbar_wait(&sb.k_empty[jk % RK], ((jk / RK) - 1) & 1, abort, p.wait_ns)) ok = false;
  if (ok) mbar_arrive(&sb.k_full[jk % RK]);
  if (ok && jv >= RV && !mbar_wait(&sb.v_empty[jv % RV], ((jv / RV) - 1) & 1, abort, p.wait_ns)) ok = false;
  if (ok) mbar_arrive(&sb.v_full[jv % RV]);
  if (nq == 0) griddep_wait();  // no copy was issued; the status word is written after the wait
  if (bad) atomicOr(p.status, kStatusBadSupport);
  if (!ok) {
    raise_status(p, &sb.abort, kStatusTimeout);
    // Let every copy already issued land before the CTA's shared memory is
    // released.
    int never = 0;
    for (int t = max(0, jk - RK); t < jk; ++t) mbar_wait(&sb.k_full[t % RK], (t / RK) & 1, &never);
    for (int t = max(0, jv - RV); t < jv; ++t) mbar_wait(&sb.v_full[t % RV], (t / RV) & 1, &never);
    if (nq > 0) mbar_wait(&sb.q_full, (nq - 1) & 1, &never);
  }
}

// --------------------------------------------------------------- MMA issuers
template <int D, int BLK, int MODE>
__device__ void attn_mma_s(const AttnParams& p, uint32_t tmem, uint8_t* q_stage, uint8_t* ring,
                           SharedState<AttnCfg<D>::kRingK, AttnCfg<D>::kRingV>& sb) {
  using C = AttnCfg<D>;
  constexpr int RK = C::kRingK;
  volatile int* abort = &sb.abort;
  constexpr uint32_t idesc_s = idesc_bf16_f32(128, kTileN, false, false);
  int j = 0, nq = 0;
  bool ok = true;
  for (;;) {
    const int slot = j % RK;
    // K(j) has landed, and with it tile j's entry of the MMA ring (written
    // before K(j) was loaded; the end marker completes the barrier without a
    // copy); S(j) overwrites S(j-1), so its softmax warpgroup must have read
    // it.  Both are probed together.
    if (!mbar_wait_both(&sb.k_full[slot], (j / RK) & 1, &sb.s_free[(j - 1) & 1], ((j - 1) >> 1) & 1, j >= 1,
                        abort, p.wait_ns)) {
      ok = false;
      break;
    }
    const int4 ent = sb.sched[kMmaRing][j % kSchedSlots];
    mbar_arrive(&sb.sched_empty[kMmaRing][j % kSchedSlots]);
    if (ent.z & kEntEnd) break;
    if (ent.z & kEntFirst) {
      // Q in TMEM was last read by the S products of unit nq - 1.
      if (nq >= 1 && !mbar_wait(&sb.q_free, (nq - 1) & 1, abort, p.wait_ns)) {
        ok = false;
        break;
      }
      if (!mbar_wait(&sb.q_full, nq & 1, abort, p.wait_ns)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint32_t q_base = smem_u32(q_stage);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk)
        tmem_cp_128x256b(tmem + C::kTmemQ + kk * 8,
                         smem_desc_sw128(q_base + (kk >> 2) * (128 * 128) + (kk & 3) * 32, 16, 1024));
      umma_commit(&sb.q_stage_free);
      ++nq;
    }
    tc_fence_after_sync();
    const uint32_t s_col = C::kTmemS;
    const uint64_t b0 = smem_desc_sw128(smem_u32(ring + slot * C::kKVBytes), 16, 1024);
#pragma unroll 1
    for (int kk = 0; kk < D / 16; ++kk) {
      // K step kk: 8 TMEM columns of Q; shared-memory descriptors of later
      // steps differ only in the start address field (address >> 4).
      const uint32_t b_off = ((kk >> 2) * (kTileN * 128) + (kk & 3) * 32) >> 4;
      umma_bf16_ts(tmem + s_col, tmem + C::kTmemQ + kk * 8, b0 + b_off, idesc_s, kk > 0 ? 1u : 0u);
    }
    umma_commit(&sb.s_full[j & 1]);
    umma_commit(&sb.k_empty[slot]);
    if (ent.z & kEntLast) umma_commit(&sb.q_free);
    ++j;
  }
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
  // Every MMA and copy issued must have completed before TMEM is released.
  umma_commit(&sb.s_done);
  int never = 0;
  mbar_wait(&sb.s_done, 0, &never);
}

template <int D, int BLK, int MODE>
__device__ void attn_mma_pv(const AttnParams& p, uint32_t tmem, uint8_t* ring,
                            SharedState<AttnCfg<D>::kRingK, AttnCfg<D>::kRingV>& sb) {
  using C = AttnCfg<D>;
  constexpr int RK = C::kRingK, RV = C::kRingV;
  uint8_t* v_ring = ring + RK * C::kKVBytes;
  volatile int* abort = &sb.abort;
  constexpr uint32_t idesc_o = idesc_bf16_f32(128, D, false, true);
  int j = 0, nu = 0;
  bool ok = true;
  for (;;) {
    const int slot = j % RV;
    // V(j) has landed, and with it tile j's entry of the MMA ring (written
    // before V(j) was loaded; the end marker completes the barrier without a
    // copy).
    if (!mbar_wait(&sb.v_full[slot], (j / RV) & 1, abort, p.wait_ns)) {
      ok = false;
      break;
    }
    const int4 ent = sb.sched[kMmaRing][j % kSchedSlots];
    mbar_arrive(&sb.sched_empty[kMmaRing][j % kSchedSlots]);
    if (ent.z & kEntEnd) break;
    const bool first = (ent.z & kEntFirst) != 0;
    if (first) {
      // The first P V of a unit overwrites O: both epilogue halves of the
      // previous unit must have read it.
      if (nu >= 1 && !mbar_wait(&sb.o_free, (nu - 1) & 1, abort, p.wait_ns)) {
        ok = false;
        break;
      }
      ++nu;
    }
    if (!mbar_wait(&sb.p_full[j & 1], (j >> 1) & 1, abort, p.wait_ns)) {
      ok = false;
      break;
    }
    tc_fence_after_sync();
    const uint32_t p_col = C::kTmemP + (j & 1) * C::kTmemPCols;
    const uint64_t b0 = smem_desc_sw128(smem_u32(v_ring + slot * C::kKVBytes), kTileN * 128, 1024);
#pragma unroll 1
    for (int kk = 0; kk < kTileN / 16; ++kk)
      umma_bf16_ts(tmem + C::kTmemO, tmem + p_col + kk * 8, b0 + ((kk * 2048) >> 4), idesc_o,
                   (first && kk == 0) ? 0u : 1u);
    umma_commit(&sb.o_full[j & 1]);
    umma_commit(&sb.v_empty[slot]);
    ++j;
  }
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
  umma_commit(&sb.pv_done);
  int never = 0;
  mbar_wait(&sb.pv_done, 0, &never);
}

// What the epilogue needs about its unit.
struct EpiInfo {
  int u;      // unit
  int j0;     // tile counter of its first tile
  int j1;     // tile counter of its last tile
  int nu;     // index among this CTA's units with tiles
  int n_kt;   // key tiles 0..n_kt-1 (dense variants)
  float l, m; // L's row-sum part and the max it refers to (the final one)
};

// ------------------------------------------------------------------- softmax
template <int D, int BLK, int MODE>
__device__ void attn_softmax(const CUtensorMap* mapO, const AttnParams& p, int w, uint32_t tmem, uint8_t* out_stage,
                             float* mass_ws,
                             SharedState<AttnCfg<D>::kRingK, AttnCfg<D>::kRingV>& sb) {
  using C = AttnCfg<D>;
  constexpr float kRescaleThreshold = 8.0f;   // log2 units: P stays <= 256
  volatile int* abort = &sb.abort;
  const int r = threadIdx.x & 127;  // query row within the tile (TMEM lane)
  const int wq = r >> 5, lane = r & 31;
  const uint32_t lane_tmem = tmem + ((uint32_t)(wq * 32) << 16);
  const uint32_t s_col = C::kTmemS;
  const uint32_t p_col = C::kTmemP + w * C::kTmemPCols;  // this warpgroup's P buffer
  constexpr int S = kTileN / BLK;   // query blocks per query tile = key blocks per key tile
  const int qsub = r / BLK;         // this row's query block within the tile
  // Per-CTA scratch (kDenseMass): log2 partial masses [2 warpgroups][2 units]
  // [key tiles / 2 + 1][S sub-blocks][128 rows] (tile t of a unit sits at
  // t / 2 in the region of the warpgroup that handled it), then
  // [2 warpgroups][2][4 warps][n_blocks] per-warp column sums.
  const int lc_tiles = p.n_qtiles / 2 + 1;
  float* cta_scratch = p.scratch + (size_t)blockIdx.x * scratch_floats_per_cta(p.n_qtiles, S, p.n_blocks);
  auto lc_at = [&](int g, int unit, int t, int k) -> float* {
    return cta_scratch + (((size_t)(g * 2 + (unit & 1)) * lc_tiles + (t >> 1)) * S + k) * 128 + r;
  };
  float* warp_sums = cta_scratch + (size_t)4 * lc_tiles * S * 128;

  int j = w;             // this warpgroup's next tile: w, w + 2, ...
  int pos = 0;           // entries read from ring w
  int n_epi = 0;         // epilogues run (as L); also the other warpgroup's publications read
  int n_pub = 0;         // publications as E
  bool fresh = true;     // the row-sum state holds no tile of the current unit
  int cur_row = 0;
  float l_w = 0.0f, m_w = -INFINITY;  // this warpgroup's part of the row sum, relative to m_w
  bool ok = true;

  // ---- one tile (j & 1 == w): key tile and mask in `key`, tile t of the
  // unit with index unit_ix
  auto tile = [&](int key, bool first, int t, int unit_ix) -> bool {
    if (!warp_wait(&sb.s_full[w], (j >> 1) & 1, abort, p.wait_ns)) return false;
    tc_fence_after_sync();
    const int kb = key & 0xFFFF;
    const uint32_t sub = ((uint32_t)key >> (16 + qsub * S)) & ((1u << S) - 1u);
    const int lim = cur_row - kb * kTileN;  // keys kb*128 + c with c > lim are in the future
    float s[kTileN];
    tmem_load_row<kTileN>(lane_tmem + s_col, s);
    // S(j) is in registers: S(j+1) may overwrite it (released before the
    // masks, which are on the path of the next S product otherwise).
    tc_fence_before_sync();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.s_free[w]);
    mask_s_row<BLK>(s, sub, lim);
    const float m_tile = row_max(s) * p.scale_log2;
    // Running max after the previous tile (the other warpgroup's).
    float m_prev = -INFINITY;
    if (!first) {
      const int jp = j - 1;
      if (!warp_wait(&sb.m_pub[w ^ 1][(jp >> 1) & 1], (jp >> 2) & 1, abort, p.wait_ns)) return false;
      m_prev = sb.mx[w ^ 1][(jp >> 1) & 1][r];
    }
    const float m_new = (m_tile > m_prev + kRescaleThreshold) ? m_tile : m_prev;
    sb.mx[w][(j >> 1) & 1][r] = m_new;
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.m_pub[w][(j >> 1) & 1]);
    float gsum[S];  // kDenseMass: sums of p over the key sub-blocks
    float rowsum;
    if constexpr (MODE == kDenseMass && S > 1) {
      rowsum = exp2_scaled_groups(s, p.scale_log2, m_new == -INFINITY ? 0.0f : m_new, gsum);
    } else {
      rowsum = exp2_scaled(s, p.scale_log2, m_new == -INFINITY ? 0.0f : m_new);
      gsum[0] = rowsum;
    }
    // P as bf16 pairs, packed before the wait below.
    uint32_t pw[kTileN / 2];
#pragma unroll
    for (int e = 0; e < kTileN / 2; ++e) pw[e] = pack_bf16x2(s[2 * e], s[2 * e + 1]);
    // P buffer w was last read by P V(j-2); this warpgroup waited for P V(j-4)
    // at its previous tile, so o_full[w] is at most one phase short.
    if (j >= 2 && !warp_wait(&sb.o_full[w], ((j >> 1) - 1) & 1, abort, p.wait_ns)) return false;
    tc_fence_after_sync();
    // The stores complete while the bookkeeping below runs.
#pragma unroll
    for (int c = 0; c < kTileN / 32; ++c) {
      uint32_t q[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) q[e] = pw[16 * c + e];
      tmem_st_32x32b_x16(lane_tmem + p_col + 16 * c, q);
    }
    if (m_new != m_w) {
      l_w *= ex2_approx(m_w - m_new);  // 0 while m_w is -inf
      m_w = m_new;
    }
    l_w += rowsum;
    // Written after the P V(j-1) wait above: tile j-1 was handled by the
    // other warpgroup after any epilogue it ran for unit unit_ix - 2 (which
    // read this slot), and this warpgroup's own epilogues precede in program
    // order.
    if constexpr (MODE == kDenseMass) {
#pragma unroll
      for (int k = 0; k < S; ++k)
        *lc_at(w, unit_ix, t, k) = gsum[k] > 0.0f ? m_new + lg2_approx(gsum[k]) : -INFINITY;
    }
    // O (after P V(j-1)) is rescaled only when the max moved.  tcgen05.ld/st
    // are warp-collective: the warp rescales together, lanes whose max did
    // not move use a factor of 1.
    const bool rescale = !first && m_new != m_prev && m_prev != -INFINITY;
    if (__any_sync(0xffffffffu, rescale)) {
      // O must have received P V(j-1); P V(j-3) completed (the wait above).
      if (!warp_wait(&sb.o_full[(j - 1) & 1], ((j - 1) >> 1) & 1, abort, p.wait_ns)) return false;
      tc_fence_after_sync();
      const float f = rescale ? ex2_approx(m_prev - m_new) : 1.0f;
#pragma unroll
      for (int c = 0; c < D / 16; ++c) {
        uint32_t v[16];
        tmem_ld_32x32b_x16(lane_tmem + C::kTmemO + 16 * c, v);
        tmem_ld_wait(v);
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * f);
        tmem_st_32x32b_x16(lane_tmem + C::kTmemO + 16 * c, v);
      }
    }
    tmem_st_wait();
    tc_fence_before_sync();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.p_full[w]);
    return true;
  };

  // ---- the epilogue, run by L (this warpgroup handled the unit's last tile)
  auto epilogue = [&](const EpiInfo& ei) -> bool {
    const int x = w ^ 1;  // E
    if (!warp_wait(&sb.l_pub[x], n_epi & 1, abort, p.wait_ns)) return false;
    const float lE = sb.lx[x][r], mE = sb.lm[x][r];
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.l_ack[x]);
    // O refers to L's max, which is the final running max; E's is at most
    // that.
    const float l_row = (mE == -INFINITY) ? ei.l : ei.l + lE * ex2_approx(mE - ei.m);
    int b, h, qt;
    decode_unit(p, ei.u, b, h, qt);
    const int row = qt * 128 + r;
    // kDenseMass: the row's first 32 partial masses (E wrote its tiles'
    // before publishing its part) and the block masses this epilogue adds to
    // are loaded now, so that their latency overlaps the wait for the last
    // P V and the output of O.  Dense variants: tile t of the unit is key
    // tile t, holding key blocks t * S .. t * S + S - 1.
    constexpr int kPrefetch = 2;  // block masses prefetched per thread
    const int n_kb = min(ei.n_kt * S, p.n_blocks);
    float v[32], prev[kPrefetch];
    auto load_lc = [&](int kb0) {
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int kb = kb0 + i, t = kb / S;
        v[i] = (kb < n_kb) ? *lc_at((ei.j0 + t) & 1, ei.nu, t, kb - t * S) : -INFINITY;
      }
    };
    // Block mass entry e (= qi * n_blocks + kb) of this unit, or null when
    // its query block lies past the end.
    auto mass_at = [&](int e) -> float* {
      const int qi = e / p.n_blocks, kb = e - qi * p.n_blocks;
      const int qblock = qt * S + qi;
      return qblock < p.n_blocks
                 ? p.blockmass + ((size_t)(b * p.n_heads + h) * p.n_blocks + qblock) * p.n_blocks + kb
                 : nullptr;
    };
    if constexpr (MODE == kDenseMass) {
      load_lc(0);
#pragma unroll
      for (int i = 0; i < kPrefetch; ++i) {
        const int e = r + 128 * i;
        float* out = (p.step > 0 && e < S * p.n_blocks && e % p.n_blocks < n_kb) ? mass_at(e) : nullptr;
        prev[i] = out ? *out : 0.0f;
      }
    }
    // P V(j1-2) completed before P(j1) was written, so o_full[j1 & 1] is at
    // most one phase short of P V(j1).
    if (!warp_wait(&sb.o_full[ei.j1 & 1], (ei.j1 >> 1) & 1, abort, p.wait_ns)) return false;
    tc_fence_after_sync();
    float o[D];
    tmem_load_row<D>(lane_tmem + C::kTmemO, o);
    tc_fence_before_sync();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.o_free);
    const float inv_l = l_row > 0.0f ? 1.0f / l_row : 0.0f;
    // O / l through this warp's staging box (32 rows x 64 columns, 128-byte
    // swizzle): each thread writes its row, then the warp reads the box back
    // four rows at a time (eight lanes per 128-byte row segment) and stores
    // it to global memory, so that each store instruction covers whole
    // segments.  Rows past seqlen and columns past D are dropped.  (TMA
    // stores from the box queue behind the K/V loads in the copy engine and
    // the box could not be refilled until they had read it.)  The epilogues
    // of consecutive units never overlap: L of a unit waits for the other
    // warpgroup's publication, which that warpgroup makes after any
    // epilogue of its own.
    uint8_t* stage = out_stage + wq * (32 * 128);
    __nv_bfloat16* o_rows = p.O + ((size_t)(b * p.n_heads + h) * p.seqlen + qt * 128 + wq * 32) * D;
    const float2 inv_l2 = make_float2(inv_l, inv_l);  // O / l two columns per packed multiply
#pragma unroll
    for (int hb = 0; hb < C::kBoxes; ++hb) {
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        const int col = hb * 64 + c * 8;
        uint32_t q[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          q[e] = 0u;
          if (col + 2 * e + 1 < D) {
            const float2 x = __fmul2_rn(make_float2(o[col + 2 * e], o[col + 2 * e + 1]), inv_l2);
            q[e] = pack_bf16x2(x.x, x.y);
          }
        }
        st_shared_v4(smem_u32(stage + lane * 128 + ((c ^ (lane & 7)) << 4)), q[0], q[1], q[2], q[3]);
      }
      __syncwarp();
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int rr = i * 4 + (lane >> 3), c = lane & 7;
        const uint4 val = ld_shared_v4(smem_u32(stage + rr * 128 + ((c ^ (rr & 7)) << 4)));
        const int col = hb * 64 + c * 8;
        if (qt * 128 + wq * 32 + rr < p.seqlen && col < D)
          *reinterpret_cast<uint4*>(o_rows + (size_t)rr * D + col) = val;
      }
      __syncwarp();
    }
    if constexpr (MODE == kDenseMass) {
      // Block mass (Eq. 5): per row 2^(lc - lse), summed over the rows of
      // each query block.
      const float lse = ei.m + lg2_approx(l_row);
      // Per-warp column sums: in shared memory when the key blocks fit
      // (double-buffered: a warp may start the next epilogue of its
      // warpgroup while another still reads this one's), else in the global
      // scratch.  The epilogues of the two warpgroups never overlap.
      const bool ws_shared = p.n_blocks <= C::kMassWsBlocks;
      const int ws_stride = ws_shared ? C::kMassWsBlocks : p.n_blocks;
      float* ws = ws_shared ? mass_ws + (n_epi & 1) * 4 * C::kMassWsBlocks
                            : warp_sums + (size_t)(w * 2 + (n_epi & 1)) * 4 * p.n_blocks;
      // 32 key blocks per pass: their partials are loaded together, and the
      // warp's 32 column sums end one per lane.
      for (int kb0 = 0; kb0 < n_kb; kb0 += 32) {
        if (kb0 > 0) load_lc(kb0);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = (row < p.seqlen) ? ex2_approx(v[i] - lse) : 0.0f;
        const float sum = warp_column_sums(v, lane);
        if (kb0 + lane < n_kb) ws[wq * ws_stride + kb0 + lane] = sum;
      }
      // Orders the four warps' writes before the reads below (release /
      // acquire at CTA scope).
      __syncwarp();
      if (lane == 0) mbar_arrive(&sb.epi[w]);
      if (!warp_wait(&sb.epi[w], n_epi & 1, abort, p.wait_ns)) return false;
      constexpr int kWarpsPerBlock = BLK / 32;  // warps holding one query block's rows
      const float inv_b = 1.0f / (float)BLK;
      for (int i = 0, e = r; e < S * p.n_blocks; ++i, e += 128) {
        const int qi = e / p.n_blocks, kb = e - qi * p.n_blocks;
        float* out = mass_at(e);
        if (!out) continue;
        if (kb < n_kb) {
          float sum = 0.0f;
#pragma unroll
          for (int q = qi * kWarpsPerBlock; q < (qi + 1) * kWarpsPerBlock; ++q) sum += ws[q * ws_stride + kb];
          sum *= inv_b;
          float before = 0.0f;
          if (p.step > 0) {
            before = i >= kPrefetch ? *out : prev[0];
#pragma unroll
            for (int k = 1; k < kPrefetch; ++k) before = (i == k) ? prev[k] : before;
          }
          *out = before + sum;
        } else if (p.step == 0) {
          *out = 0.0f;
        }
      }
    }
    ++n_epi;
    return true;
  };

  // ---- E's publication of its part of the row sum for the unit that just
  // ended (zero if this warpgroup handled none of its tiles), once L has read
  // the previous one.
  auto publish = [&]() -> bool {
    if (n_pub >= 1 && !warp_wait(&sb.l_ack[w], (n_pub - 1) & 1, abort, p.wait_ns)) return false;
    sb.lx[w][r] = fresh ? 0.0f : l_w;
    sb.lm[w][r] = fresh ? -INFINITY : m_w;
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.l_pub[w]);
    ++n_pub;
    fresh = true;
    return true;
  };

  for (;;) {
    const int slot = pos % kSchedSlots;
    if (!warp_wait(&sb.sched_full[w][slot], (pos / kSchedSlots) & 1, abort, p.wait_ns)) {
      ok = false;
      break;
    }
    const int4 ent = sb.sched[w][slot];
    __syncwarp();
    if (lane == 0) mbar_arrive(&sb.sched_empty[w][slot]);
    ++pos;
    const int fl = ent.z;
    if (fl & kEntEnd) {
      // The last unit ended at tile ent.w - 1; if the other warpgroup handled
      // it, this one is that unit's E.
      if (ent.w >= 1 && ((ent.w - 1) & 1) != w && !publish()) ok = false;
      break;
    }
    if (fl & kEntEmpty) {
      // No key tile (ring 0 only): the rows of the unit attend nothing and
      // are zero.
      int b, h, qt;
      decode_unit(p, ent.y, b, h, qt);
      const int row = qt * 128 + r;
      if (row < p.seqlen) {
        uint4* dst = reinterpret_cast<uint4*>(p.O + ((size_t)(b * p.n_heads + h) * p.seqlen + row) * D);
#pragma unroll
        for (int c = 0; c < D / 8; ++c) dst[c] = make_uint4(0u, 0u, 0u, 0u);
      }
      continue;
    }
    const bool first = (fl & kEntFirst) != 0;
    // Tile j - 1 (the other warpgroup's) ended the previous unit: this
    // warpgroup is that unit's E.
    if (first && j >= 1 && !publish()) {
      ok = false;
      break;
    }
    if (fresh) {
      int b, h, qt;
      decode_unit(p, ent.y, b, h, qt);
      cur_row = qt * 128 + r;
      l_w = 0.0f;
      m_w = -INFINITY;
    }
    if (!tile(ent.x, first, ent.w, fl >> kEntUnitShift)) {
      ok = false;
      break;
    }
    fresh = false;
    if (fl & kEntLast) {
      // L: this warpgroup handled the unit's last tile.
      const EpiInfo ei{ent.y, j - ent.w, j, fl >> kEntUnitShift, (ent.x & 0xFFFF) + 1, l_w, m_w};
      if (!epilogue(ei)) {
        ok = false;
        break;
      }
      fresh = true;
    }
    j += 2;
  }
  // A warp that gave up inside a tile may still have TMEM stores in flight:
  // they complete before TMEM is released.  Output stores issued by this
  // warp complete before the CTA exits.
  tmem_st_wait();
  if (lane == 0) tma_store_wait_all();
  if (!ok) raise_status(p, &sb.abort, kStatusTimeout);
}

// -------------------------------------------------------------------- kernel
template <int D, int BLK, int MODE>
__global__ void __launch_bounds__(AttnCfg<D>::kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                const __grid_constant__ CUtensorMap mapV, const __grid_constant__ CUtensorMap mapO,
                const AttnParams p) {
  using C = AttnCfg<D>;
  using SS = SharedState<C::kRingK, C::kRingV>;
  static_assert(sizeof(SS) <= C::kStaticReserve, "static shared memory");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* q_stage = smem;             // one Q tile
  uint8_t* ring = smem + C::kQBytes;   // kRing K/V entries
  uint8_t* out_stage = ring + C::kRing * C::kKVBytes;  // epilogue staging (1024-byte aligned), then the
                                                       // block-mass column sums
  __shared__ SS sb;

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
    for (int i = 0; i < kSchedSlots; ++i) {
      for (int rw = 0; rw < 3; ++rw) {
        mbar_init(&sb.sched_full[rw][i], 1);
        mbar_init(&sb.sched_empty[rw][i], rw == kMmaRing ? 2 : 4);  // its readers
      }
    }
    mbar_init(&sb.q_full, 1);
    mbar_init(&sb.q_stage_free, 1);
    mbar_init(&sb.q_free, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&sb.s_full[b], 1);
      mbar_init(&sb.s_free[b], 4);
      mbar_init(&sb.p_full[b], 4);
      mbar_init(&sb.m_pub[b][0], 4);
      mbar_init(&sb.m_pub[b][1], 4);
      mbar_init(&sb.l_pub[b], 4);
      mbar_init(&sb.l_ack[b], 4);
      mbar_init(&sb.epi[b], 4);
      mbar_init(&sb.o_full[b], 1);
    }
    mbar_init(&sb.o_free, 4);
    for (int b = 0; b < kStageSlots; ++b) {
      mbar_init(&sb.list_full[b], 1);
      mbar_init(&sb.list_empty[b], 1);
    }
    mbar_init(&sb.s_done, 1);
    mbar_init(&sb.pv_done, 1);
    fence_mbar_init();
  }
  if (warp == C::kProducerWarp && lane == 0) {
    tma_prefetch_map(&mapQ);
    tma_prefetch_map(&mapK);
    tma_prefetch_map(&mapV);
    tma_prefetch_map(&mapO);
  }
  if (warp == C::kMmaSWarp) {
    tmem_alloc(&sb.tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sb.tmem_base;
  // Set-up above touched no global memory: with a programmatic launch it
  // overlaps the tail of the previous kernel of the stream.  Every access to
  // Q, K, V, O and blockmass comes after the wait; the producer and the
  // schedule stager may read idx and counts before it (the only kernels
  // that launch this one early are attention kernels, which write O and
  // blockmass only), so the producer waits just before its first copy.  The
  // next kernel may then be scheduled; its CTAs take SMs as this grid's CTAs
  // exit.
  if (warp != C::kProducerWarp && warp != 11) griddep_wait();
  if (threadIdx.x == 0) griddep_launch_dependents();

  if (warp < 8) {
    warpgroup_reg_inc<C::kRegsSoftmax>();
    attn_softmax<D, BLK, MODE>(&mapO, p, warp >> 2, tmem, out_stage,
                               reinterpret_cast<float*>(out_stage + C::kOutBytes), sb);
  } else {
    warpgroup_reg_dec<C::kRegsOther>();
    if (warp == C::kProducerWarp) {
      if (lane == 0) attn_producer<D, BLK, MODE>(&mapQ, &mapK, &mapV, p, q_stage, ring, sb);
    } else if (warp == C::kMmaSWarp) {
      if (lane == 0) attn_mma_s<D, BLK, MODE>(p, tmem, q_stage, ring, sb);
    } else if (warp == C::kMmaPVWarp) {
      if (lane == 0) attn_mma_pv<D, BLK, MODE>(p, tmem, ring, sb);
    } else if (sched_staging<BLK, MODE>(p)) {
      attn_sched_stager<D, BLK, MODE>(p, sb);  // warp 11
    }
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

template <int D, int BLK, int MODE>
cudaError_t launch_attn_instance(const AttnLaunch& L) {
  using C = AttnCfg<D>;
  auto kern = attn_kernel<D, BLK, MODE>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemLaunch);
  if (e != cudaSuccess) return e;
  // Programmatic stream serialization: the grid may be scheduled while the
  // previous kernel of the stream finishes (see griddep_wait in the kernel).
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(L.grid);
  cfg.blockDim = dim3(C::kThreads);
  cfg.dynamicSmemBytes = C::kSmemLaunch;
  cfg.stream = L.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, L.mapQ, L.mapK, L.mapV, L.mapO, L.p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_attn_for_dim(int block, int mode, const AttnLaunch& L) {
  // Plain dense attention does not depend on the block size (every sub-block
  // is attended, causality is applied per row).
  if (mode == kDense) return launch_attn_instance<D, 128, kDense>(L);
  switch (block) {
    case 128:
      return mode == kDenseMass ? launch_attn_instance<D, 128, kDenseMass>(L) : launch_attn_instance<D, 128, kSparse>(L);
    case 64:
      return mode == kDenseMass ? launch_attn_instance<D, 64, kDenseMass>(L) : launch_attn_instance<D, 64, kSparse>(L);
    default:
      return mode == kDenseMass ? launch_attn_instance<D, 32, kDenseMass>(L) : launch_attn_instance<D, 32, kSparse>(L);
  }
}

}  // namespace wise
