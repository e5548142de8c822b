// Routing diagnostics: the block attention mass of a step retained by a
// support, and the overlap of two supports (rolling-set Jaccard).
#include <limits.h>

#include "internal.cuh"

namespace wise {
namespace {

// One thread per query-head row (b, h, q): the row's masses r_qb summed over
// the key blocks of its kv-group's support list, in list order.  Entries that
// are negative, beyond the query block, or not strictly above the previous
// accepted entry are skipped (the attention kernels' rule) and reported.
__global__ void __launch_bounds__(256) support_mass_kernel(const SupportMassParams p) {
  const long long row = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (row >= p.rows) return;
  const int q = (int)(row % p.n_blocks);
  const long long bh = row / p.n_blocks;
  const int h = (int)(bh % p.n_heads);
  const int b = (int)(bh / p.n_heads);
  const long long srow = ((long long)b * p.n_kv_heads + h / p.group) * p.n_blocks + q;
  int n = __ldg(p.counts + srow);
  int bad = 0;
  if (n < 0 || n > p.cap) {
    bad = 1;
    n = n < 0 ? 0 : p.cap;
  }
  const int32_t* list = p.idx + srow * p.cap;
  const float* m = p.blockmass + row * p.n_blocks;
  float acc = 0.0f;
  int prev = -1;
  for (int i = 0; i < n; ++i) {
    const int v = __ldg(list + i);
    if (v >= 0 && v <= q && v > prev) {
      acc += __ldg(m + v);
      prev = v;
    } else {
      bad = 1;
    }
  }
  p.retained[row] = acc;
  if (bad) atomicOr(p.status, kStatusBadSupport);
}

// Next entry of a support list that the attention kernels use (in [0, q] and
// strictly above the last accepted one), or INT_MAX when the list is done.
__device__ __forceinline__ int next_valid(const int32_t* list, int n, int q, int& i, int& prev, int& bad) {
  while (i < n) {
    const int v = __ldg(list + i);
    ++i;
    if (v >= 0 && v <= q && v > prev) {
      prev = v;
      return v;
    }
    bad = 1;
  }
  return INT_MAX;
}

__device__ __forceinline__ int clamp_list(int n, int cap, int& bad) {
  if (n < 0 || n > cap) {
    bad = 1;
    return n < 0 ? 0 : cap;
  }
  return n;
}

// One CTA per batch element; each thread merges the two (ascending) lists of
// its rows (b, kv head, q) and counts the blocks in both and in either.  The
// counts are integers, so the result does not depend on the reduction order.
__global__ void __launch_bounds__(256) support_overlap_kernel(const SupportOverlapParams p) {
  const int b = blockIdx.x;
  unsigned long long inter = 0, uni = 0;
  int bad = 0;
  for (int r = threadIdx.x; r < p.rows; r += blockDim.x) {
    const long long row = (long long)b * p.rows + r;
    const int q = r % p.n_blocks;
    const int na = clamp_list(__ldg(p.counts_a + row), p.cap_a, bad);
    const int nb = clamp_list(__ldg(p.counts_b + row), p.cap_b, bad);
    const int32_t* la = p.idx_a + row * p.cap_a;
    const int32_t* lb = p.idx_b + row * p.cap_b;
    int ia = 0, ib = 0, pa = -1, pb = -1;
    int va = next_valid(la, na, q, ia, pa, bad), vb = next_valid(lb, nb, q, ib, pb, bad);
    while (va != INT_MAX || vb != INT_MAX) {
      ++uni;
      if (va == vb) {
        ++inter;
        va = next_valid(la, na, q, ia, pa, bad);
        vb = next_valid(lb, nb, q, ib, pb, bad);
      } else if (va < vb) {
        va = next_valid(la, na, q, ia, pa, bad);
      } else {
        vb = next_valid(lb, nb, q, ib, pb, bad);
      }
    }
  }
  __shared__ unsigned long long part[2][8];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    inter += __shfl_xor_sync(0xffffffffu, inter, off);
    uni += __shfl_xor_sync(0xffffffffu, uni, off);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    part[0][warp] = inter;
    part[1][warp] = uni;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long ti = 0, tu = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      ti += part[0][w];
      tu += part[1][w];
    }
    p.inter_union[2 * b] = ti;
    p.inter_union[2 * b + 1] = tu;
  }
  if (bad) atomicOr(p.status, kStatusBadSupport);
}

}  // namespace

cudaError_t launch_support_overlap(const SupportOverlapParams& p, cudaStream_t stream) {
  support_overlap_kernel<<<p.batch, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_support_mass(const SupportMassParams& p, cudaStream_t stream) {
  const long long blocks = (p.rows + 255) / 256;
  support_mass_kernel<<<(unsigned)blocks, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace wise
