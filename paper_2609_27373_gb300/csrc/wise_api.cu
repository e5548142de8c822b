// Host side of the C ABI declared in include/wise.h: argument checks, TMA
// tensor maps, the per-device scratch buffer and status word, and launches.
#include <limits.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <math.h>
#include <mutex>

#include "wise.h"
#include "internal.cuh"
#include "ptx.cuh"

namespace wise {
namespace {

// Per-device status word; kernels OR kStatus* bits into it.
__device__ int g_status;

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool probed = false;
  bool supported = false;
  int sm_count = 0;
  int* status = nullptr;  // device address of g_status
  float* scratch = nullptr;
  size_t scratch_bytes = 0;
};

std::mutex g_mutex;
DeviceState g_dev[kMaxDevices];

// Limit of each bounded wait inside the attention kernels, taken by every
// later launch (wise_set_wait_limit_ns).
std::atomic<unsigned long long> g_wait_ns{kWaitLimitNs};

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// Current device's state, probing it on first use.  Returns nullptr (and sets
// *err) when there is no usable device.
DeviceState* device_state(int* err) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *err = WISE_ERR_CUDA;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState& s = g_dev[dev];
  if (!s.probed) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      *err = WISE_ERR_CUDA;
      return nullptr;
    }
    s.supported = (major == 10 && minor == 3);  // the library is built for sm_103a only
    s.sm_count = sms;
    if (s.supported && cudaGetSymbolAddress(reinterpret_cast<void**>(&s.status), g_status) != cudaSuccess) {
      *err = WISE_ERR_CUDA;
      return nullptr;
    }
    s.probed = true;
  }
  if (!s.supported) {
    *err = WISE_ERR_UNSUPPORTED;
    return nullptr;
  }
  return &s;
}

// Grows the device's scratch buffer to at least `bytes`.  Frees the previous
// buffer first (cudaFree waits for the device to be idle).
float* scratch_at_least(DeviceState* s, size_t bytes) {
  std::lock_guard<std::mutex> lock(g_mutex);
  if (s->scratch_bytes >= bytes) return s->scratch;
  if (s->scratch) cudaFree(s->scratch);
  s->scratch = nullptr;
  s->scratch_bytes = 0;
  if (cudaMalloc(reinterpret_cast<void**>(&s->scratch), bytes) != cudaSuccess) {
    s->scratch = nullptr;
    return nullptr;
  }
  s->scratch_bytes = bytes;
  return s->scratch;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_shape(const wise_shape_t* sh, bool attention) {
  if (!sh) return WISE_ERR_INVALID_ARG;
  if (sh->batch < 0 || sh->seqlen < 0 || sh->n_heads <= 0 || sh->n_kv_heads <= 0 || sh->block <= 0 ||
      sh->head_dim <= 0 || !(sh->scale >= 0.0f) || isinf(sh->scale))
    return WISE_ERR_INVALID_ARG;
  if (sh->n_heads % sh->n_kv_heads != 0) return WISE_ERR_UNSUPPORTED;
  if (sh->block != 32 && sh->block != 64 && sh->block != 128) return WISE_ERR_UNSUPPORTED;
  if (attention && sh->head_dim != 64 && sh->head_dim != 96 && sh->head_dim != 128) return WISE_ERR_UNSUPPORTED;
  if (sh->seqlen % sh->block != 0) return WISE_ERR_SHAPE;
  if ((long long)sh->batch * sh->n_heads > (1LL << 24)) return WISE_ERR_UNSUPPORTED;
  if ((long long)sh->seqlen > (1LL << 20)) return WISE_ERR_UNSUPPORTED;
  return WISE_OK;
}

// Tensor map over a [rows_outer, seqlen, head_dim] bf16 array with 64-column,
// box_rows-row boxes in the 128-byte swizzle.  Rows past seqlen read as zero
// and are not written by stores.
bool make_map(CUtensorMap* map, const void* base, int head_dim, int seqlen, long long outer, int box_rows) {
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)head_dim, (cuuint64_t)seqlen, (cuuint64_t)outer};
  cuuint64_t strides[2] = {(cuuint64_t)head_dim * 2, (cuuint64_t)head_dim * 2 * (cuuint64_t)seqlen};
  cuuint32_t box[3] = {64, (cuuint32_t)box_rows, 1};
  cuuint32_t elem[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, elem,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

int launch_attention(const wise_shape_t* sh, const void* Q, const void* K, const void* V, void* O, int mode,
                     float* blockmass, int step, const int32_t* idx, const int32_t* counts, int cap,
                     cudaStream_t stream, bool fixed_scratch) {
  int rc = check_shape(sh, true);
  if (rc != WISE_OK) return rc;
  if (sh->batch == 0 || sh->seqlen == 0) return WISE_OK;
  if (!Q || !K || !V || !O || !aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(O, 16))
    return WISE_ERR_INVALID_ARG;
  const int n_blocks = sh->seqlen / sh->block;
  if (mode == kDenseMass) {
    if (!aligned(blockmass, 4) || step < 0) return WISE_ERR_INVALID_ARG;
  }
  if (mode == kSparse) {
    if (!idx || !counts || !aligned(idx, 4) || !aligned(counts, 4) || cap <= 0) return WISE_ERR_INVALID_ARG;
    if (cap > 65535) return WISE_ERR_UNSUPPORTED;
  }
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;

  AttnLaunch L;
  const long long outer_q = (long long)sh->batch * sh->n_heads;
  const long long outer_kv = (long long)sh->batch * sh->n_kv_heads;
  if (!make_map(&L.mapQ, Q, sh->head_dim, sh->seqlen, outer_q, 128) ||
      !make_map(&L.mapK, K, sh->head_dim, sh->seqlen, outer_kv, 128) ||
      !make_map(&L.mapV, V, sh->head_dim, sh->seqlen, outer_kv, 128) ||
      !make_map(&L.mapO, O, sh->head_dim, sh->seqlen, outer_q, 32))
    return WISE_ERR_CUDA;

  AttnParams& p = L.p;
  p.batch = sh->batch;
  p.seqlen = sh->seqlen;
  p.n_heads = sh->n_heads;
  p.n_kv_heads = sh->n_kv_heads;
  p.group = sh->n_heads / sh->n_kv_heads;
  p.n_qtiles = (sh->seqlen + 127) / 128;
  p.n_blocks = n_blocks;
  const long long units = outer_q * p.n_qtiles;
  if (units > INT32_MAX) return WISE_ERR_UNSUPPORTED;
  p.n_units = (int)units;
  // Unit order: when the K and V of all heads do not stay resident in L2
  // (more than 64 MiB), heads are processed in equal groups of whole kv-head
  // groups whose K and V take at most 48 MiB, so that each K/V tile is read
  // from DRAM about once instead of once per wave of query tiles.
  {
    const double kv_bytes = (double)sh->seqlen * sh->head_dim * 2.0 * 2.0;  // K and V of one kv head
    p.group_heads = 0;
    if (kv_bytes * (double)outer_kv > 64.0 * (1 << 20)) {
      long long g_kv = (long long)((48.0 * (1 << 20)) / kv_bytes);
      if (g_kv < 1) g_kv = 1;
      const long long n_groups = (outer_kv + g_kv - 1) / g_kv;
      g_kv = (outer_kv + n_groups - 1) / n_groups;
      p.group_heads = (int)(g_kv * p.group);
    }
  }
  const float scale = sh->scale > 0.0f ? sh->scale : 1.0f / sqrtf((float)sh->head_dim);
  p.scale_log2 = scale * 1.4426950408889634f;
  p.O = reinterpret_cast<__nv_bfloat16*>(O);
  p.blockmass = blockmass;
  p.step = step;
  p.idx = idx;
  p.counts = counts;
  p.cap = cap;
  p.status = ds->status;
  p.wait_ns = g_wait_ns.load(std::memory_order_relaxed);
  L.grid = (int)(units < ds->sm_count ? units : ds->sm_count);
  L.stream = stream;
  p.scratch = nullptr;
  if (mode == kDenseMass) {
    // Per CTA: log2 partial masses per key sub-block and per-warp sums.
    const size_t need =
        (size_t)L.grid * scratch_floats_per_cta(p.n_qtiles, 128 / sh->block, n_blocks) * sizeof(float);
    if (fixed_scratch) {
      if (need > WISE_NOALLOC_SCRATCH_BYTES) return WISE_ERR_UNSUPPORTED;
      const int rs = noalloc_scratch_address(&p.scratch);
      if (rs != WISE_OK) return rs;
    } else {
      p.scratch = scratch_at_least(ds, need);
      if (!p.scratch) return WISE_ERR_CUDA;
    }
  }
  cudaError_t e;
  switch (sh->head_dim) {
    case 64: e = launch_attn_d64(sh->block, mode, L); break;
    case 96: e = launch_attn_d96(sh->block, mode, L); break;
    default: e = launch_attn_d128(sh->block, mode, L); break;
  }
  return e == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

}  // namespace wise

using namespace wise;

extern "C" int wise_full_attn_accumulate(const wise_shape_t* shape, const void* Q, const void* K, const void* V,
                                         void* O, float* blockmass, int step, cudaStream_t stream) {
  return launch_attention(shape, Q, K, V, O, blockmass ? kDenseMass : kDense, blockmass, step, nullptr, nullptr,
                          0, stream);
}

extern "C" int wise_sparse_attn(const wise_shape_t* shape, const void* Q, const void* K, const void* V,
                                const int32_t* idx, const int32_t* counts, int cap, void* O, cudaStream_t stream) {
  return launch_attention(shape, Q, K, V, O, kSparse, nullptr, 0, idx, counts, cap, stream);
}

extern "C" int wise_freeze_a_attn(const wise_shape_t* shape, const void* Q_frozen, const void* K_frozen,
                                  const void* V, const int32_t* idx, const int32_t* counts, int cap, void* O,
                                  cudaStream_t stream) {
  // The frozen distribution restricted to the support and renormalised is the
  // softmax over the support of the frozen step's logits, so the sparse kernel
  // computes it from that step's Q and K against the current V.
  return launch_attention(shape, Q_frozen, K_frozen, V, O, kSparse, nullptr, 0, idx, counts, cap, stream);
}

namespace {

// Shared checks and parameters of the two stored-distribution calls.
int freeze_setup(const wise_shape_t* sh, const int32_t* idx, const int32_t* counts, int cap, const void* P,
                 const float* inv_l, int tile_cap, FreezeLaunch& L) {
  int rc = check_shape(sh, true);
  if (rc != WISE_OK) return rc;
  if (cap <= 0 || !P || !aligned(P, 16) || !inv_l || !aligned(inv_l, 4)) return WISE_ERR_INVALID_ARG;
  if (cap > 65535) return WISE_ERR_UNSUPPORTED;
  if (sh->batch == 0 || sh->seqlen == 0) return WISE_OK;
  if (!idx || !counts || !aligned(idx, 4) || !aligned(counts, 4)) return WISE_ERR_INVALID_ARG;
  const int n_qtiles = (sh->seqlen + 127) / 128;
  const long long walk_max = std::min<long long>(n_qtiles, (long long)(128 / sh->block) * cap);
  if (tile_cap < walk_max) return WISE_ERR_INVALID_ARG;
  const long long units = (long long)sh->batch * sh->n_heads * n_qtiles;
  if (units * tile_cap > INT32_MAX) return WISE_ERR_UNSUPPORTED;
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  AttnParams& p = L.p;
  memset(&p, 0, sizeof(p));
  p.batch = sh->batch;
  p.seqlen = sh->seqlen;
  p.n_heads = sh->n_heads;
  p.n_kv_heads = sh->n_kv_heads;
  p.group = sh->n_heads / sh->n_kv_heads;
  p.n_qtiles = n_qtiles;
  p.n_blocks = sh->seqlen / sh->block;
  p.n_units = (int)units;
  const float scale = sh->scale > 0.0f ? sh->scale : 1.0f / sqrtf((float)sh->head_dim);
  p.scale_log2 = scale * 1.4426950408889634f;
  p.idx = idx;
  p.counts = counts;
  p.cap = cap;
  p.status = ds->status;
  L.P = reinterpret_cast<__nv_bfloat16*>(const_cast<void*>(P));
  L.inv_l = const_cast<float*>(inv_l);
  L.tile_cap = tile_cap;
  return WISE_OK;
}

}  // namespace

extern "C" int wise_freeze_a_probs(const wise_shape_t* shape, const void* Q_frozen, const void* K_frozen,
                                   const int32_t* idx, const int32_t* counts, int cap, void* P, float* inv_l,
                                   int tile_cap, cudaStream_t stream) {
  FreezeLaunch L;
  int rc = freeze_setup(shape, idx, counts, cap, P, inv_l, tile_cap, L);
  if (rc != WISE_OK || shape->batch == 0 || shape->seqlen == 0) return rc;
  if (!Q_frozen || !K_frozen || !aligned(Q_frozen, 16) || !aligned(K_frozen, 16)) return WISE_ERR_INVALID_ARG;
  const long long outer_q = (long long)shape->batch * shape->n_heads;
  const long long outer_kv = (long long)shape->batch * shape->n_kv_heads;
  if (!make_map(&L.mapQ, Q_frozen, shape->head_dim, shape->seqlen, outer_q, 128) ||
      !make_map(&L.mapK, K_frozen, shape->head_dim, shape->seqlen, outer_kv, 128))
    return WISE_ERR_CUDA;
  L.stream = stream;
  return launch_freeze_probs(shape->head_dim, shape->block, L) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_frozen_pv(const wise_shape_t* shape, const void* P, const float* inv_l, int tile_cap,
                              const void* V, const int32_t* idx, const int32_t* counts, int cap, void* O,
                              cudaStream_t stream) {
  FreezeLaunch L;
  int rc = freeze_setup(shape, idx, counts, cap, P, inv_l, tile_cap, L);
  if (rc != WISE_OK || shape->batch == 0 || shape->seqlen == 0) return rc;
  if (!V || !O || !aligned(V, 16) || !aligned(O, 16)) return WISE_ERR_INVALID_ARG;
  const long long outer_kv = (long long)shape->batch * shape->n_kv_heads;
  if (!make_map(&L.mapV, V, shape->head_dim, shape->seqlen, outer_kv, 128) ||
      !make_map(&L.mapP, P, 128, 128, (long long)L.p.n_units * tile_cap, 128))
    return WISE_ERR_CUDA;
  L.p.O = reinterpret_cast<__nv_bfloat16*>(O);
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  L.grid = L.p.n_units < ds->sm_count ? L.p.n_units : ds->sm_count;
  L.stream = stream;
  return launch_frozen_pv(shape->head_dim, shape->block, L) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_select_support(const wise_shape_t* shape, const wise_select_t* sel, const float* blockmass,
                                   int32_t* idx, int32_t* counts, cudaStream_t stream) {
  int rc = check_shape(shape, false);
  if (rc != WISE_OK) return rc;
  if (!sel) return WISE_ERR_INVALID_ARG;
  if (sel->n_sink < 0 || sel->n_local < 1 || sel->cap < sel->n_sink + sel->n_local) return WISE_ERR_INVALID_ARG;
  if (sel->mode != WISE_SEL_TOPK && sel->mode != WISE_SEL_COVERAGE) return WISE_ERR_INVALID_ARG;
  if (sel->mode == WISE_SEL_TOPK && sel->topk < 0) return WISE_ERR_INVALID_ARG;
  if (sel->mode == WISE_SEL_COVERAGE && !(sel->eta >= 0.0f && sel->eta <= 1.0f)) return WISE_ERR_INVALID_ARG;
  if (shape->batch == 0 || shape->seqlen == 0) return WISE_OK;
  const int n_blocks = shape->seqlen / shape->block;
  if (n_blocks > 1024) return WISE_ERR_UNSUPPORTED;
  if (!blockmass || !idx || !counts || !aligned(blockmass, 4) || !aligned(idx, 4) || !aligned(counts, 4))
    return WISE_ERR_INVALID_ARG;
  int err = WISE_OK;
  if (!device_state(&err)) return err;
  SelectParams p;
  p.batch = shape->batch;
  p.n_heads = shape->n_heads;
  p.n_kv_heads = shape->n_kv_heads;
  p.group = shape->n_heads / shape->n_kv_heads;
  p.n_blocks = n_blocks;
  p.n_sink = sel->n_sink;
  p.n_local = sel->n_local;
  p.mode = sel->mode;
  p.topk = sel->topk;
  p.cap = sel->cap;
  p.eta16 = (uint64_t)floor((double)sel->eta * 65536.0 + 0.5);
  p.blockmass = blockmass;
  p.idx = idx;
  p.counts = counts;
  return launch_select(p, stream) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_select_working_set(const wise_shape_t* shape, int mode, float eta, int n_sink, int n_local,
                                       const float* step_masses, int n_steps, const int32_t* ref_idx,
                                       const int32_t* ref_counts, int ref_cap, int32_t* idx, int32_t* counts,
                                       int cap, cudaStream_t stream) {
  int rc = check_shape(shape, false);
  if (rc != WISE_OK) return rc;
  if (mode < WISE_WS_UNION || mode > WISE_WS_SIZE_MATCHED) return WISE_ERR_INVALID_ARG;
  if (n_sink < 0 || n_local < 0) return WISE_ERR_INVALID_ARG;
  if (mode <= WISE_WS_STATIC && !(eta >= 0.0f && eta <= 1.0f)) return WISE_ERR_INVALID_ARG;
  if (mode == WISE_WS_UNION ? n_steps < 1 : n_steps != 1) return WISE_ERR_INVALID_ARG;
  const int n_blocks = shape->seqlen / shape->block;
  if (shape->batch == 0 || shape->seqlen == 0) return WISE_OK;
  if (n_blocks > 1024) return WISE_ERR_UNSUPPORTED;
  if (cap < n_blocks) return WISE_ERR_INVALID_ARG;
  if (!step_masses || !idx || !counts || !aligned(step_masses, 4) || !aligned(idx, 4) || !aligned(counts, 4))
    return WISE_ERR_INVALID_ARG;
  if (mode >= WISE_WS_MASS_MATCHED &&
      (!ref_idx || !ref_counts || ref_cap <= 0 || !aligned(ref_idx, 4) || !aligned(ref_counts, 4)))
    return WISE_ERR_INVALID_ARG;
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  WorkingSetParams p;
  p.batch = shape->batch;
  p.n_heads = shape->n_heads;
  p.n_kv_heads = shape->n_kv_heads;
  p.group = shape->n_heads / shape->n_kv_heads;
  p.n_blocks = n_blocks;
  p.n_sink = n_sink;
  p.n_local = n_local;
  p.mode = mode;
  p.n_steps = n_steps;
  p.cap = cap;
  p.ref_cap = mode >= WISE_WS_MASS_MATCHED ? ref_cap : 1;
  p.eta16 = (uint64_t)floor((double)eta * 65536.0 + 0.5);
  p.masses = step_masses;
  p.ref_idx = ref_idx;
  p.ref_counts = ref_counts;
  p.idx = idx;
  p.counts = counts;
  p.status = ds->status;
  return launch_working_set(p, stream) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_support_mass(const wise_shape_t* shape, const float* blockmass, const int32_t* idx,
                                 const int32_t* counts, int cap, float* retained, cudaStream_t stream) {
  int rc = check_shape(shape, false);
  if (rc != WISE_OK) return rc;
  if (cap <= 0) return WISE_ERR_INVALID_ARG;
  if (shape->batch == 0 || shape->seqlen == 0) return WISE_OK;
  if (!blockmass || !idx || !counts || !retained || !aligned(blockmass, 4) || !aligned(idx, 4) ||
      !aligned(counts, 4) || !aligned(retained, 4))
    return WISE_ERR_INVALID_ARG;
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  SupportMassParams p;
  p.n_heads = shape->n_heads;
  p.n_kv_heads = shape->n_kv_heads;
  p.group = shape->n_heads / shape->n_kv_heads;
  p.n_blocks = shape->seqlen / shape->block;
  p.rows = (long long)shape->batch * shape->n_heads * p.n_blocks;
  p.cap = cap;
  p.blockmass = blockmass;
  p.idx = idx;
  p.counts = counts;
  p.retained = retained;
  p.status = ds->status;
  return launch_support_mass(p, stream) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_support_overlap(const wise_shape_t* shape, const int32_t* idx_a, const int32_t* counts_a,
                                    int cap_a, const int32_t* idx_b, const int32_t* counts_b, int cap_b,
                                    unsigned long long* inter_union, cudaStream_t stream) {
  int rc = check_shape(shape, false);
  if (rc != WISE_OK) return rc;
  if (cap_a <= 0 || cap_b <= 0) return WISE_ERR_INVALID_ARG;
  if (shape->batch == 0) return WISE_OK;
  if (!inter_union || !aligned(inter_union, 8)) return WISE_ERR_INVALID_ARG;
  const long long rows = (long long)shape->n_kv_heads * (shape->seqlen / shape->block);
  if (rows > INT_MAX) return WISE_ERR_UNSUPPORTED;
  if (rows > 0 && (!idx_a || !counts_a || !idx_b || !counts_b || !aligned(idx_a, 4) || !aligned(counts_a, 4) ||
                   !aligned(idx_b, 4) || !aligned(counts_b, 4)))
    return WISE_ERR_INVALID_ARG;
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  SupportOverlapParams p;
  p.batch = shape->batch;
  p.rows = (int)rows;
  p.n_blocks = shape->seqlen / shape->block;
  p.cap_a = cap_a;
  p.cap_b = cap_b;
  p.idx_a = idx_a;
  p.counts_a = counts_a;
  p.idx_b = idx_b;
  p.counts_b = counts_b;
  p.inter_union = inter_union;
  p.status = ds->status;
  return launch_support_overlap(p, stream) == cudaSuccess ? WISE_OK : WISE_ERR_CUDA;
}

extern "C" int wise_get_status(cudaStream_t stream) {
  int err = WISE_OK;
  DeviceState* ds = device_state(&err);
  if (!ds) return err;
  if (cudaStreamSynchronize(stream) != cudaSuccess) return WISE_ERR_CUDA;
  int word = 0;
  if (cudaMemcpyFromSymbol(&word, g_status, sizeof(int)) != cudaSuccess) return WISE_ERR_CUDA;
  if (word) {
    const int zero = 0;
    if (cudaMemcpyToSymbol(g_status, &zero, sizeof(int)) != cudaSuccess) return WISE_ERR_CUDA;
  }
  if (word & kStatusTimeout) return WISE_ERR_TIMEOUT;
  if (word & kStatusBadSupport) return WISE_ERR_BAD_SUPPORT;
  return WISE_OK;
}

extern "C" const char* wise_status_string(int status) {
  switch (status) {
    case WISE_OK: return "ok";
    case WISE_ERR_INVALID_ARG: return "invalid argument (null, misaligned, negative size or bad selection rule)";
    case WISE_ERR_UNSUPPORTED: return "unsupported configuration (head_dim, block, head grouping or device)";
    case WISE_ERR_SHAPE: return "seqlen is not a multiple of block";
    case WISE_ERR_CUDA: return "CUDA runtime error";
    case WISE_ERR_TIMEOUT: return "a kernel wait ran out of time";
    case WISE_ERR_BAD_SUPPORT: return "support list entries out of range, unordered or over cap";
    default: return "unknown status";
  }
}

extern "C" int wise_set_wait_limit_ns(unsigned long long ns) {
  g_wait_ns.store(ns == 0 ? kWaitLimitNs : ns, std::memory_order_relaxed);
  return WISE_OK;
}

extern "C" int wise_version(void) { return 100; }
