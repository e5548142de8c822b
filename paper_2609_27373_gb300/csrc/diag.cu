// Routing diagnostic: block attention mass of a step retained by a support.
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

}  // namespace

cudaError_t launch_support_mass(const SupportMassParams& p, cudaStream_t stream) {
  const long long blocks = (p.rows + 255) / 256;
  support_mass_kernel<<<(unsigned)blocks, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace wise
