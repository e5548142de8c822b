// Support selection (Eq. 6, single-pass form over accumulated block mass).
//
// One warp per (batch, kv-head, query block) row.  Lane l owns key blocks
// l, l + 32, ... (KPL of them).  Masses of the kv-head group's query heads are
// pooled in exact 64-bit fixed point, the forced sink/local blocks are marked,
// and the remaining admissible blocks are taken one at a time in rank order
// (pooled mass descending, block index ascending) by a warp-wide argmax over
// shuffles, until top-k is reached or the kept mass covers eta of the row's
// admissible mass (cum * 65536 >= eta16 * total, compared in 128 bits), never
// beyond `cap`.  The chosen set is written in ascending order with ballots and
// prefix popcounts, padded with -1.
#include <limits.h>

#include "internal.cuh"

namespace wise {

__device__ __forceinline__ uint64_t mass_units(float x) {
  if (!(x > 0.0f)) return 0ull;  // negative, zero and NaN masses count as zero
  x = fminf(x, 4096.0f);
  return __double2ull_rz(floor(static_cast<double>(x) * 4294967296.0));
}

__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// cum * 65536 < eta16 * total, exactly.
__device__ __forceinline__ bool below_threshold(uint64_t cum, uint64_t eta16, uint64_t total) {
  const uint64_t lhs_hi = cum >> 48, lhs_lo = cum << 16;
  const uint64_t rhs_hi = __umul64hi(eta16, total), rhs_lo = eta16 * total;
  return lhs_hi < rhs_hi || (lhs_hi == rhs_hi && lhs_lo < rhs_lo);
}

template <int KPL>
__global__ void __launch_bounds__(256) select_kernel(const SelectParams p) {
  const long row = (long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const long n_rows = (long)p.batch * p.n_kv_heads * p.n_blocks;
  if (row >= n_rows) return;
  const int lane = threadIdx.x & 31;
  const int nb = p.n_blocks;
  const int q = (int)(row % nb);
  const int g = (int)((row / nb) % p.n_kv_heads);
  const int b = (int)(row / ((long)nb * p.n_kv_heads));

  uint64_t U[KPL];
  uint32_t cand = 0, chosen = 0;  // bit i <-> block lane + 32 i
  uint64_t total_part = 0, cum_part = 0;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    const int kb = lane + 32 * i;
    U[i] = 0;
    if (kb <= q) {
      for (int h = g * p.group; h < (g + 1) * p.group; ++h)
        U[i] += mass_units(__ldg(p.blockmass + (((size_t)b * p.n_heads + h) * nb + q) * nb + kb));
      total_part += U[i];
      const bool forced = kb < p.n_sink || kb > q - p.n_local;
      if (forced) {
        chosen |= 1u << i;
        cum_part += U[i];
      } else {
        cand |= 1u << i;
      }
    }
  }
  const uint64_t total = warp_sum_u64(total_part);
  uint64_t cum = warp_sum_u64(cum_part);
  int n = 0;
#pragma unroll
  for (int i = 0; i < KPL; ++i) n += __popc(__ballot_sync(0xffffffffu, (chosen >> i) & 1u));

  const int budget = (p.mode == 0) ? min(p.topk, p.cap - n) : p.cap - n;
  for (int t = 0; t < budget; ++t) {
    if (p.mode != 0 && !below_threshold(cum, p.eta16, total)) break;
    // Best candidate of this lane: larger mass first, then lower block.
    uint64_t best_u = 0;
    int best_kb = INT_MAX;
#pragma unroll
    for (int i = 0; i < KPL; ++i) {
      if (((cand >> i) & 1u) && (best_kb == INT_MAX || U[i] > best_u)) {
        best_u = U[i];
        best_kb = lane + 32 * i;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const uint64_t ou = __shfl_xor_sync(0xffffffffu, best_u, off);
      const int okb = __shfl_xor_sync(0xffffffffu, best_kb, off);
      const bool take = (okb != INT_MAX) && (best_kb == INT_MAX || ou > best_u || (ou == best_u && okb < best_kb));
      if (take) {
        best_u = ou;
        best_kb = okb;
      }
    }
    if (best_kb == INT_MAX) break;  // no candidate left
    if ((best_kb & 31) == lane) {
      const uint32_t bit = 1u << (best_kb >> 5);
      cand &= ~bit;
      chosen |= bit;
    }
    cum += best_u;
    ++n;
  }

  int32_t* out = p.idx + row * p.cap;
  int base = 0;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    const uint32_t ball = __ballot_sync(0xffffffffu, (chosen >> i) & 1u);
    if ((chosen >> i) & 1u) out[base + __popc(ball & ((1u << lane) - 1u))] = lane + 32 * i;
    base += __popc(ball);
  }
  for (int pos = n + lane; pos < p.cap; pos += 32) out[pos] = -1;
  if (lane == 0) p.counts[row] = n;
}

template <int KPL>
static cudaError_t launch_select_kpl(const SelectParams& p, cudaStream_t stream) {
  const long rows = (long)p.batch * p.n_kv_heads * p.n_blocks;
  const int warps = 8;
  const long grid = (rows + warps - 1) / warps;
  select_kernel<KPL><<<(unsigned)grid, warps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_select(const SelectParams& p, cudaStream_t stream) {
  if (p.n_blocks <= 32) return launch_select_kpl<1>(p, stream);
  if (p.n_blocks <= 64) return launch_select_kpl<2>(p, stream);
  if (p.n_blocks <= 128) return launch_select_kpl<4>(p, stream);
  if (p.n_blocks <= 256) return launch_select_kpl<8>(p, stream);
  if (p.n_blocks <= 512) return launch_select_kpl<16>(p, stream);
  return launch_select_kpl<32>(p, stream);
}

// ----------------------------------------------------------- working sets
// wise_select_working_set: the paper's own working set and its controls,
// one warp per (batch, kv-head, query block) row, same fixed-point masses,
// ranking and exact threshold comparison as select_kernel, no cap (the host
// requires cap >= nKB).  Modes: 0 union of per-step eta coverage sets (Eq. 6
// with the window union), 1 static (the first step's eta coverage set),
// 2 mass matched, 3 size matched (first step's ranking against a reference
// working set).  Forced sink/local blocks belong to every set.

// Warp-wide best remaining candidate: larger mass first, then lower block.
template <int KPL>
__device__ __forceinline__ int ws_argmax(const uint64_t (&U)[KPL], uint32_t cand, int lane, uint64_t& best_u) {
  best_u = 0;
  int best_kb = INT_MAX;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    if (((cand >> i) & 1u) && (best_kb == INT_MAX || U[i] > best_u)) {
      best_u = U[i];
      best_kb = lane + 32 * i;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const uint64_t ou = __shfl_xor_sync(0xffffffffu, best_u, off);
    const int okb = __shfl_xor_sync(0xffffffffu, best_kb, off);
    const bool take = (okb != INT_MAX) && (best_kb == INT_MAX || ou > best_u || (ou == best_u && okb < best_kb));
    if (take) {
      best_u = ou;
      best_kb = okb;
    }
  }
  return best_kb;
}

// Pooled fixed-point masses of one step for this lane's blocks.
template <int KPL>
__device__ __forceinline__ void ws_pool(const WorkingSetParams& p, int step, int b, int g, int q, int lane,
                                        uint64_t (&U)[KPL]) {
  const int nb = p.n_blocks;
  const float* m = p.masses + (size_t)step * p.batch * p.n_heads * nb * nb;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    const int kb = lane + 32 * i;
    U[i] = 0;
    if (kb <= q)
      for (int h = g * p.group; h < (g + 1) * p.group; ++h)
        U[i] += mass_units(__ldg(m + (((size_t)b * p.n_heads + h) * nb + q) * nb + kb));
  }
}

// Adds candidates in rank order to `chosen` (mass cum) until stop(cum) or
// `budget` additions or no candidate is left.
template <int KPL, class Stop>
__device__ __forceinline__ void ws_take(const uint64_t (&U)[KPL], uint32_t& cand, uint32_t& chosen, uint64_t& cum,
                                        int budget, int lane, Stop stop) {
  for (int t = 0; t < budget; ++t) {
    if (stop(cum)) break;
    uint64_t best_u;
    const int best_kb = ws_argmax(U, cand, lane, best_u);
    if (best_kb == INT_MAX) break;
    if ((best_kb & 31) == lane) {
      const uint32_t bit = 1u << (best_kb >> 5);
      cand &= ~bit;
      chosen |= bit;
    }
    cum += best_u;
  }
}

template <int KPL>
__global__ void __launch_bounds__(256) working_set_kernel(const WorkingSetParams p) {
  const long row = (long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const long n_rows = (long)p.batch * p.n_kv_heads * p.n_blocks;
  if (row >= n_rows) return;
  const int lane = threadIdx.x & 31;
  const int nb = p.n_blocks;
  const int q = (int)(row % nb);
  const int g = (int)((row / nb) % p.n_kv_heads);
  const int b = (int)(row / ((long)nb * p.n_kv_heads));

  uint32_t admissible = 0, forced = 0;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    const int kb = lane + 32 * i;
    if (kb <= q) {
      admissible |= 1u << i;
      if (kb < p.n_sink || kb > q - p.n_local) forced |= 1u << i;
    }
  }
  uint64_t U[KPL];
  uint32_t result = forced;
  if (p.mode <= 1) {
    // Union over the steps of each step's eta coverage set (one step: static).
    for (int st = 0; st < p.n_steps; ++st) {
      ws_pool(p, st, b, g, q, lane, U);
      uint64_t total_part = 0, cum_part = 0;
#pragma unroll
      for (int i = 0; i < KPL; ++i) {
        if ((admissible >> i) & 1u) total_part += U[i];
        if ((forced >> i) & 1u) cum_part += U[i];
      }
      const uint64_t total = warp_sum_u64(total_part);
      uint64_t cum = warp_sum_u64(cum_part);
      uint32_t cand = admissible & ~forced, chosen = forced;
      ws_take(U, cand, chosen, cum, nb, lane,
              [&](uint64_t c) { return !below_threshold(c, p.eta16, total); });
      result |= chosen;
    }
  } else {
    // The reference working set of this row: its size and its first-step mass.
    ws_pool(p, 0, b, g, q, lane, U);
    const int32_t* ref = p.ref_idx + row * p.ref_cap;
    int n_ref = __ldg(p.ref_counts + row);
    int bad = 0;
    if (n_ref < 0 || n_ref > p.ref_cap) {
      bad = 1;
      n_ref = n_ref < 0 ? 0 : p.ref_cap;
    }
    uint32_t in_ref = 0;
    int prev = -1, k_ref = 0;
    for (int e = 0; e < n_ref; ++e) {
      const int v = __ldg(ref + e);  // the same value for every lane
      if (v >= 0 && v <= q && v > prev) {
        prev = v;
        ++k_ref;
        if ((v & 31) == lane) in_ref |= 1u << (v >> 5);
      } else {
        bad = 1;
      }
    }
    if (bad && lane == 0) atomicOr(p.status, kStatusBadSupport);
    uint64_t ref_part = 0, cum_part = 0;
    int n_forced_part = 0;
#pragma unroll
    for (int i = 0; i < KPL; ++i) {
      if ((in_ref >> i) & 1u) ref_part += U[i];
      if ((forced >> i) & 1u) {
        cum_part += U[i];
        ++n_forced_part;
      }
    }
    const uint64_t target = warp_sum_u64(ref_part);
    uint64_t cum = warp_sum_u64(cum_part);
    int n_forced = n_forced_part;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) n_forced += __shfl_xor_sync(0xffffffffu, n_forced, off);
    uint32_t cand = admissible & ~forced, chosen = forced;
    if (p.mode == 2)
      ws_take(U, cand, chosen, cum, nb, lane, [&](uint64_t c) { return c >= target; });
    else
      ws_take(U, cand, chosen, cum, k_ref - n_forced, lane, [](uint64_t) { return false; });
    result = chosen;
  }

  int32_t* out = p.idx + row * p.cap;
  int base = 0;
#pragma unroll
  for (int i = 0; i < KPL; ++i) {
    const uint32_t ball = __ballot_sync(0xffffffffu, (result >> i) & 1u);
    if ((result >> i) & 1u) out[base + __popc(ball & ((1u << lane) - 1u))] = lane + 32 * i;
    base += __popc(ball);
  }
  for (int pos = base + lane; pos < p.cap; pos += 32) out[pos] = -1;
  if (lane == 0) p.counts[row] = base;
}

template <int KPL>
static cudaError_t launch_ws_kpl(const WorkingSetParams& p, cudaStream_t stream) {
  const long rows = (long)p.batch * p.n_kv_heads * p.n_blocks;
  const int warps = 8;
  const long grid = (rows + warps - 1) / warps;
  working_set_kernel<KPL><<<(unsigned)grid, warps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_working_set(const WorkingSetParams& p, cudaStream_t stream) {
  if (p.n_blocks <= 32) return launch_ws_kpl<1>(p, stream);
  if (p.n_blocks <= 64) return launch_ws_kpl<2>(p, stream);
  if (p.n_blocks <= 128) return launch_ws_kpl<4>(p, stream);
  if (p.n_blocks <= 256) return launch_ws_kpl<8>(p, stream);
  if (p.n_blocks <= 512) return launch_ws_kpl<16>(p, stream);
  return launch_ws_kpl<32>(p, stream);
}

}  // namespace wise
