// Declarations shared by the translation units of libwise.so.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "wise.h"

namespace wise {

enum AttnMode : int { kDense = 0, kDenseMass = 1, kSparse = 2 };

// Per-CTA scratch of kDenseMass, in floats, for n_tiles key tiles of 128
// keys holding sub key blocks each (n_blocks key blocks in all): log2 partial
// masses [2 warpgroups][2 units][n_tiles / 2 + 1][sub][128 rows] (a
// warpgroup handles every other tile of a unit, and keeps the previous unit's
// values until its epilogue has read them), then per-warp column sums
// [2 warpgroups][2][4 warps][n_blocks] (used only when the kernel's shared
// memory copy of them, for up to 128 key blocks, is too small).
__host__ __device__ constexpr size_t scratch_floats_per_cta(int n_tiles, int sub, int n_blocks) {
  return (size_t)512 * sub * (n_tiles / 2 + 1) + (size_t)16 * n_blocks;
}

// Bits of the per-device status word.
constexpr int kStatusTimeout = 1;
constexpr int kStatusBadSupport = 2;

struct AttnParams {
  int batch, seqlen, n_heads, n_kv_heads, group;
  int n_qtiles;   // ceil(seqlen / 128): 128-row query tiles
  int n_blocks;   // nQB = nKB = seqlen / block
  int n_units;    // batch * n_heads * n_qtiles
  int group_heads;  // unit order (decode_unit): 0 = by query tile over all heads, else heads in groups of this size
  float scale_log2;
  __nv_bfloat16* O;
  float* blockmass;       // kDenseMass
  int step;               // kDenseMass: 0 overwrites, > 0 accumulates
  const int32_t* idx;     // kSparse
  const int32_t* counts;  // kSparse
  int cap;                // kSparse
  float* scratch;         // kDenseMass: scratch_floats_per_cta(n_blocks) floats per CTA
  int* status;
  unsigned long long wait_ns;  // limit of each bounded wait on the main path (kWaitLimitNs by default)
};

struct AttnLaunch {
  CUtensorMap mapQ, mapK, mapV;
  CUtensorMap mapO;  // output, 32-row boxes (TMA stores of the epilogue)
  AttnParams p;
  int grid;
  cudaStream_t stream;
};

// Defined in attn_d64.cu / attn_d96.cu / attn_d128.cu.
cudaError_t launch_attn_d64(int block, int mode, const AttnLaunch& L);
cudaError_t launch_attn_d96(int block, int mode, const AttnLaunch& L);
cudaError_t launch_attn_d128(int block, int mode, const AttnLaunch& L);

struct SelectParams {
  int batch, n_heads, n_kv_heads, group, n_blocks;
  int n_sink, n_local, mode, topk, cap;
  uint64_t eta16;  // floor(eta * 65536 + 0.5)
  const float* blockmass;
  int32_t* idx;
  int32_t* counts;
};

// Argument checks, tensor maps and launch of the attention kernels (defined
// in wise_api.cu).  For kDenseMass the per-CTA scratch comes from the
// library's lazily allocated per-device buffer, unless fixed_scratch is set:
// then it is the fixed array of noalloc.cu (its address resolved by
// noalloc_scratch_address once the arguments and the device have been
// checked), and a problem needing more than WISE_NOALLOC_SCRATCH_BYTES
// returns WISE_ERR_UNSUPPORTED.
int launch_attention(const wise_shape_t* sh, const void* Q, const void* K, const void* V, void* O, int mode,
                     float* blockmass, int step, const int32_t* idx, const int32_t* counts, int cap,
                     cudaStream_t stream, bool fixed_scratch = false);

// Device address of the fixed scratch array on the current device (looked up
// once per device and cached; defined in noalloc.cu).
int noalloc_scratch_address(float** out);

// Defined in select.cu.
cudaError_t launch_select(const SelectParams& p, cudaStream_t stream);

// Working-set construction of the paper's own form and its controls
// (wise_select_working_set).
struct WorkingSetParams {
  int batch, n_heads, n_kv_heads, group, n_blocks;
  int n_sink, n_local, mode, n_steps, cap, ref_cap;
  uint64_t eta16;           // floor(eta * 65536 + 0.5)
  const float* masses;      // [n_steps][batch][n_heads][nQB][nKB]
  const int32_t* ref_idx;   // reference working set (mass / size matched)
  const int32_t* ref_counts;
  int32_t* idx;
  int32_t* counts;
  int* status;
};

// Defined in select.cu.
cudaError_t launch_working_set(const WorkingSetParams& p, cudaStream_t stream);

struct SupportMassParams {
  long long rows;  // batch * n_heads * n_blocks
  int n_heads, n_kv_heads, group, n_blocks, cap;
  const float* blockmass;
  const int32_t* idx;
  const int32_t* counts;
  float* retained;
  int* status;
};

// Freeze-A with a stored distribution (freeze.cu).  For unit u (the 128-row
// query tile qt of (b, h), u = (b * n_heads + h) * n_qtiles + qt) and the
// t-th key tile of its support walk, P + ((u * tile_cap + t) * 128 + row) * 128
// holds the bf16 tile of 2^(s - m_row); inv_l[u * 128 + row] = 1 / (row sum),
// so that Abar = diag(inv_l) P.
struct FreezeLaunch {
  CUtensorMap mapQ, mapK;  // wise_freeze_a_probs: the frozen step's Q and K (128-row boxes)
  CUtensorMap mapV, mapP;  // wise_frozen_pv: current V, and P viewed as [tiles][128][128]
  AttnParams p;            // shape, support lists, scale, status; O for wise_frozen_pv
  __nv_bfloat16* P;
  float* inv_l;
  int tile_cap;
  int grid;  // wise_frozen_pv: persistent grid, min(n_units, SM count)
  cudaStream_t stream;
};
cudaError_t launch_freeze_probs(int head_dim, int block, const FreezeLaunch& L);
cudaError_t launch_frozen_pv(int head_dim, int block, const FreezeLaunch& L);

struct SupportOverlapParams {
  int batch, rows;  // rows per batch element: n_kv_heads * n_blocks
  int n_blocks, cap_a, cap_b;
  const int32_t* idx_a;
  const int32_t* counts_a;
  const int32_t* idx_b;
  const int32_t* counts_b;
  unsigned long long* inter_union;  // [batch][2]
  int* status;
};

// Defined in diag.cu.
cudaError_t launch_support_mass(const SupportMassParams& p, cudaStream_t stream);
cudaError_t launch_support_overlap(const SupportOverlapParams& p, cudaStream_t stream);

}  // namespace wise
