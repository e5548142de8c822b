/*
 * wise.h -- C ABI of the WISE attention hot path on GB300 (sm_103a).
 *
 * WISE (working-set inference with support exploitation) runs a
 * recurrent-depth transformer's attention in two phases (Sec. 5):
 *   discovery  dense causal attention (Eq. 2) whose block attention mass
 *              (Eq. 5) is accumulated over the early recurrent steps;
 *   selection  the accumulated mass is turned, once, into a per-(batch,
 *              kv-head, query-block) list of key blocks (Eq. 6);
 *   reuse      late steps recompute Q, K, V and the softmax, restricted to
 *              that fixed block support (Eqs. 7-8).
 * Each entry point below is one hand-written CUDA kernel.
 *
 * Conventions shared by all entry points
 *  - Tensors are dense, contiguous, row-major device buffers owned by the
 *    caller.  Q and O are [batch, n_heads, seqlen, head_dim] bf16; K and V are
 *    [batch, n_kv_heads, seqlen, head_dim] bf16.  Query head h reads kv-head
 *    h / (n_heads / n_kv_heads) (grouped-query attention).
 *  - Q/K/V/O must be 16-byte aligned, blockmass/idx/counts 4-byte aligned.
 *  - head_dim is 64, 96 or 128; block (B) is 32 (the paper's default, Sec.
 *    5.1), 64 or 128; seqlen % block == 0.  nQB = nKB = seqlen / block.  The
 *    attention kernels compute 128 x 128 tiles whatever B is: a smaller block
 *    is a sub-block of a tile, masked per (query block, key block) pair.
 *  - Every call is asynchronous on `stream` and returns a status code
 *    (WISE_OK or a negative WISE_ERR_*) describing argument checks and the
 *    launch; nothing is done when a check fails.  Faults found by a kernel
 *    while it runs (an inconsistent support list, an internal wait that ran
 *    out) are recorded in a per-device status word read by wise_get_status().
 *  - Empty problems (batch == 0 or seqlen == 0) return WISE_OK and launch
 *    nothing.
 *  - The attention calls (wise_full_attn_accumulate and its _noalloc variant,
 *    wise_sparse_attn, wise_freeze_a_attn) are launched as programmatic
 *    dependents: their set-up, and their reads of idx and counts, may overlap
 *    the end of the preceding attention call on the same stream, whose other
 *    effects they wait for.  So idx and counts must not share memory with the
 *    O or blockmass of the preceding attention call.
 *  - Inputs are never written.  The library keeps one lazily allocated
 *    scratch buffer per device for the block-mass epilogue (see
 *    wise_full_attn_accumulate); no other call allocates device memory.
 */
#ifndef WISE_H_
#define WISE_H_

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define WISE_OK 0
#define WISE_ERR_INVALID_ARG -1 /* NULL or misaligned pointer, negative size, bad selection parameters */
#define WISE_ERR_UNSUPPORTED -2 /* head_dim / block / head grouping / device not supported */
#define WISE_ERR_SHAPE -3       /* seqlen not a multiple of block */
#define WISE_ERR_CUDA -4        /* a CUDA runtime call or kernel launch failed */
#define WISE_ERR_TIMEOUT -5     /* a kernel's internal wait ran out (reported by wise_get_status) */
#define WISE_ERR_BAD_SUPPORT -6 /* idx/counts held entries outside the rules (reported by wise_get_status) */

#define WISE_SEL_TOPK 0
#define WISE_SEL_COVERAGE 1

/* Modes of wise_select_working_set. */
#define WISE_WS_UNION 0
#define WISE_WS_STATIC 1
#define WISE_WS_MASS_MATCHED 2
#define WISE_WS_SIZE_MATCHED 3

/* Problem geometry (Sec. 3: n = seqlen, d_h = head_dim; Sec. 5.1: block B). */
typedef struct {
  int batch;
  int seqlen;
  int n_heads;    /* query heads */
  int n_kv_heads; /* key/value heads; n_heads % n_kv_heads == 0 */
  int head_dim;
  int block;
  float scale;    /* softmax scale; 0 selects 1/sqrt(head_dim) as in Eq. 2 */
} wise_shape_t;

/* Support-selection rule (Eq. 6, single-pass form).
 * For query block q the admissible key blocks are 0..q.  Forced blocks:
 * 0..n_sink-1 and q-n_local+1..q (clipped to 0..q).  The remaining blocks are
 * ranked by pooled fixed-point mass (descending; ties to the lower index) and
 * added in rank order:
 *   WISE_SEL_TOPK      the first `topk` of them;
 *   WISE_SEL_COVERAGE  until the kept mass reaches eta of the admissible
 *                      mass (the cumulative-mass support of Eq. 6);
 * never exceeding `cap` blocks in total, forced ones included. */
typedef struct {
  int n_sink;  /* >= 0 */
  int n_local; /* >= 1 (1 = diagonal block only) */
  int mode;    /* WISE_SEL_TOPK or WISE_SEL_COVERAGE */
  int topk;    /* >= 0, used by WISE_SEL_TOPK */
  float eta;   /* in [0, 1], used by WISE_SEL_COVERAGE */
  int cap;     /* >= n_sink + n_local; width of each idx row */
} wise_select_t;

/* Dense causal attention of one recurrent step, with the block attention
 * mass of that step accumulated on the fly.
 *   O = softmax(Q K^T * scale + M) V, M causal                      (Eq. 2)
 *   r_qb = (1/B) sum_{i in I_q} sum_{j in I_b} A_ij                  (Eq. 5)
 *   blockmass[b,h,q,kb] = (step == 0 ? 0 : blockmass[b,h,q,kb]) + r_qkb
 * blockmass is fp32 [batch, n_heads, nQB, nKB] (per query head; entries with
 * kb > q are written as 0 when step == 0 and left as they are otherwise).
 * blockmass == NULL runs plain dense attention (the dense baseline) and
 * ignores `step`.  Accumulation with step > 0 is a read-modify-write: calls on
 * the same blockmass must be ordered on the stream.
 * The first call with blockmass != NULL on a device allocates the library's
 * scratch buffer (and grows it when a later shape needs more); make that
 * first call outside any CUDA-graph capture. */
int wise_full_attn_accumulate(const wise_shape_t* shape, const void* Q, const void* K, const void* V, void* O,
                              float* blockmass, int step, cudaStream_t stream);

/* Capacity of the fixed scratch array used by
 * wise_full_attn_accumulate_noalloc (8 MiB per device). */
#define WISE_NOALLOC_SCRATCH_BYTES (8u << 20)

/* wise_full_attn_accumulate with a non-NULL blockmass, for callers that
 * cannot have this library allocate device memory.  The paper has no
 * counterpart: this is a deployment variant of the same kernel.
 *
 * Who needs it: a process whose device memory is handed out by another
 * allocator (a framework's caching allocator that has reserved the pool, a
 * fixed memory budget), or a serving loop that cannot afford the device-wide
 * synchronisation cudaMalloc/cudaFree may cause while other streams run.
 * wise_full_attn_accumulate obtains its scratch with cudaMalloc on first use
 * (and frees and reallocates it when a larger problem comes); this entry
 * point calls neither cudaMalloc nor cudaFree nor any allocating routine.
 * Its scratch is a fixed array of WISE_NOALLOC_SCRATCH_BYTES compiled into
 * the library, held by every device that loads the library until the
 * process exits.
 *
 * Arguments, layouts and results are those of wise_full_attn_accumulate;
 * blockmass must not be NULL (plain dense attention uses no scratch).
 * Limit: with nT = ceil(seqlen/128) tiles and S = 128/block, one call needs
 * min(batch*n_heads*nT, SM count) * (2048 * S * (nT/2 + 1) + 64 * nKB)
 * bytes of scratch (nT/2 rounded down); larger problems return
 * WISE_ERR_UNSUPPORTED and launch nothing.  On a 152-SM GB300 with at least
 * 152 query tiles that is nT <= 49 with block 128 (seqlen <= 6272).
 * The first call on each device that passes the argument checks looks up
 * the array's device address (with that device current) and caches it; make
 * that first call before any CUDA stream capture.  The cached address is not
 * refreshed: calls must not span a cudaDeviceReset of the device.  All calls
 * on a device share the one array: calls whose kernels can run at the same
 * time on that device (unordered streams) race on it and corrupt each other's
 * block mass.  Argument checks and error codes are those of
 * wise_full_attn_accumulate (blockmass == NULL is WISE_ERR_INVALID_ARG). */
int wise_full_attn_accumulate_noalloc(const wise_shape_t* shape, const void* Q, const void* K, const void* V,
                                      void* O, float* blockmass, int step, cudaStream_t stream);

/* Support selection from accumulated block mass (Eq. 6, rule of
 * wise_select_t).  Masses of the query heads of each kv-head group are pooled
 * in exact fixed point, u(x) = floor(min(x, 4096) * 2^32) for x > 0 (else 0),
 * so the result is a deterministic function of the fp32 input; coverage
 * compares cum * 65536 >= floor(eta * 65536 + 0.5) * total exactly.
 * blockmass: fp32 [batch, n_heads, nQB, nKB], entries kb <= q are read.
 * idx:    int32 [batch, n_kv_heads, nQB, cap], ascending block ids, -1 padded.
 * counts: int32 [batch, n_kv_heads, nQB]. */
int wise_select_support(const wise_shape_t* shape, const wise_select_t* sel, const float* blockmass,
                        int32_t* idx, int32_t* counts, cudaStream_t stream);

/* Working sets of the paper's own form and its intervention controls
 * (Eq. 6 with the union over the discovery window; appendix "Experimental
 * details", intervention controls).  Per (batch, kv head, query block q),
 * on the masses of the group's query heads pooled in the fixed point of
 * wise_select_support, with admissible blocks 0..q ranked by pooled mass
 * (descending, then block index ascending), forced blocks
 * F = {0..n_sink-1} U {q-n_local+1..q} in every set, and a coverage set
 * C_t(eta) = F plus candidates in rank order until the kept mass reaches eta
 * of the admissible mass of step t:
 *   WISE_WS_UNION         union of C_t(eta) over the n_steps given steps
 *                         (the paper: steps t_d-3..t_d, eta = 0.95, F empty)
 *   WISE_WS_STATIC        C_0(eta) of the one step given (Static-95)
 *   WISE_WS_MASS_MATCHED  F plus candidates of the one step given until the
 *                         kept mass reaches that step's mass inside the
 *                         reference set (MassMatched)
 *   WISE_WS_SIZE_MATCHED  F plus the top candidates of the one step given up
 *                         to the reference set's size (SizeMatched)
 * step_masses: fp32 [n_steps][batch][n_heads][nQB][nKB], each step's own
 * block mass (Eq. 5, wise_full_attn_accumulate with step 0).  n_steps must
 * be 1 except for WISE_WS_UNION.  ref_idx / ref_counts (row width ref_cap):
 * the reference working set for the matched controls (ignored otherwise;
 * invalid entries are skipped and reported as WISE_ERR_BAD_SUPPORT by
 * wise_get_status).  idx / counts as wise_select_support's, with row width
 * cap >= nKB (these sets have no size bound).  n_sink, n_local >= 0. */
int wise_select_working_set(const wise_shape_t* shape, int mode, float eta, int n_sink, int n_local,
                            const float* step_masses, int n_steps, const int32_t* ref_idx,
                            const int32_t* ref_counts, int ref_cap, int32_t* idx, int32_t* counts, int cap,
                            cudaStream_t stream);

/* Routing diagnostic (appendix "Experimental details", evaluation metrics:
 * retained future attention mass).  For every query-head row (b, h, q):
 *   retained[b][h][q] = sum over the key blocks kb of the support list of
 *                       the kv-group of h of blockmass[b][h][q][kb]
 * With blockmass = one step's mass (wise_full_attn_accumulate with step 0 on
 * that step's Q, K, V, i.e. Eq. 5 of the unrestricted attention), this is the
 * fraction of the step's full attention that the frozen support keeps (1 for
 * a support holding every admissible block).
 * blockmass: fp32 [batch, n_heads, nQB, nKB]; idx, counts: as produced by
 * wise_select_support (row width `cap`); retained: fp32 [batch, n_heads, nQB],
 * written.  The sum is fp32 in list order (deterministic).  List entries that
 * are negative, beyond the query block, or not strictly ascending are skipped
 * and reported as WISE_ERR_BAD_SUPPORT by wise_get_status. */
int wise_support_mass(const wise_shape_t* shape, const float* blockmass, const int32_t* idx, const int32_t* counts,
                      int cap, float* retained, cudaStream_t stream);

/* Attention of one late recurrent step restricted to the block support
 *   R_ij = 0 if b(j) in B_q(i) else -inf                              (Eq. 7)
 *   O = softmax(Q K^T * scale + M + R) V, M causal                    (Eq. 8)
 * Q, K, V are the current step's (recomputed every step, Sec. 5.2); idx and
 * counts are wise_select_support's output (row width `cap`).  Query head h
 * uses the support of kv-head h / (n_heads / n_kv_heads).  Within each row the
 * first counts entries are used; they must be ascending block ids in
 * [0, q].  Entries that break this are skipped and flagged as
 * WISE_ERR_BAD_SUPPORT in the status word.  A query row with no admissible key
 * gets O = 0.  cap <= 0 is WISE_ERR_INVALID_ARG, cap > 65535
 * WISE_ERR_UNSUPPORTED. */
int wise_sparse_attn(const wise_shape_t* shape, const void* Q, const void* K, const void* V, const int32_t* idx,
                     const int32_t* counts, int cap, void* O, cudaStream_t stream);

/* Freeze-A control (appendix "Experimental details", intervention controls):
 * the support W of WISE, with the within-support attention distribution frozen
 * at a past step t0 (the discovery endpoint):
 *   Abar_ij = A(t0)_ij [b(j) in W_q(i)] / sum_k A(t0)_ik [b(k) in W_q(i)],
 *   O = Abar V,
 * where A(t0) is that step's unrestricted causal attention and V the current
 * step's values.  The full-attention normaliser cancels in Abar, so Abar is
 * the softmax of scale * Q(t0) K(t0)^T + M + R over the support (Eqs. 7-8 with
 * the frozen Q and K): Q_frozen and K_frozen are step t0's queries and keys,
 * V the current values, all in the layouts of wise_sparse_attn, which this
 * call runs; idx, counts, cap, O, errors and the treatment of malformed lists
 * as there. */
int wise_freeze_a_attn(const wise_shape_t* shape, const void* Q_frozen, const void* K_frozen, const void* V,
                       const int32_t* idx, const int32_t* counts, int cap, void* O, cudaStream_t stream);

/* Freeze-A with a stored distribution, step 1 of 2: computes Abar of the
 * frozen step once (definition above wise_freeze_a_attn) and stores it as
 * Abar = P diag(inv_l).  With S = 128 / block, each 128-row query tile
 * u = (b * n_heads + h) * ceil(seqlen / 128) + qt walks the 128-key tiles that
 * hold blocks of its S query blocks' support lists, in ascending order; for
 * the t-th of them, P + ((u * tile_cap + t) * 128 + row) * 128 holds the
 * 128 x 128 bf16 tile of 2^(s - m_row) (row = query row, column = key within
 * the tile; m_row the row's maximum logit over the support, so its largest
 * entry is 1; exactly 0 where masked), and inv_l[u * 128 + row] = 1 / (sum of
 * the row's entries), 0 for a row without an admissible key.
 * P: device, n_units * tile_cap * 32 KiB, 16-byte aligned (tiles past a
 * unit's walk are left as they are); inv_l: device fp32, n_units * 128,
 * 4-byte aligned.  tile_cap >= min(ceil(seqlen / 128), S * cap), else
 * WISE_ERR_INVALID_ARG.  Q_frozen, K_frozen, idx, counts and cap as in
 * wise_sparse_attn. */
int wise_freeze_a_probs(const wise_shape_t* shape, const void* Q_frozen, const void* K_frozen, const int32_t* idx,
                        const int32_t* counts, int cap, void* P, float* inv_l, int tile_cap, cudaStream_t stream);

/* Freeze-A with a stored distribution, step 2 of 2, once per late step:
 *   O = Abar V = diag(inv_l) P V
 * from P and inv_l as wise_freeze_a_probs stored them (same shape, idx,
 * counts, cap and tile_cap) and the current step's V; a block-sparse P V
 * product that reads the stored tiles from HBM.  O layout as in
 * wise_sparse_attn; units without a tile give O = 0. */
int wise_frozen_pv(const wise_shape_t* shape, const void* P, const float* inv_l, int tile_cap, const void* V,
                   const int32_t* idx, const int32_t* counts, int cap, void* O, cudaStream_t stream);

/* Overlap of two block supports A and B (e.g. the rolling working sets of two
 * consecutive steps, appendix "Stability of the Deployed Working Set"): for
 * each batch element e, over all (kv head, query block) rows,
 *   inter_union[2e]     = number of (row, key block) pairs in both A and B,
 *   inter_union[2e + 1] = number in A or B,
 * so that the element's rolling-set Jaccard is inter / union (defined as 1
 * when both are empty).  idx_a/counts_a (row width cap_a) and idx_b/counts_b
 * (row width cap_b): layouts of wise_select_support's output.  inter_union:
 * device, 2 * batch unsigned 64-bit integers, 8-byte aligned, overwritten.
 * Exact integer counts.  List entries are used as the attention kernels use
 * them: malformed entries are skipped and flagged as WISE_ERR_BAD_SUPPORT.
 * Errors: INVALID_ARG for NULL or misaligned pointers or a cap <= 0; the shape
 * rules of wise_select_support (head_dim unused). */
int wise_support_overlap(const wise_shape_t* shape, const int32_t* idx_a, const int32_t* counts_a, int cap_a,
                         const int32_t* idx_b, const int32_t* counts_b, int cap_b, unsigned long long* inter_union,
                         cudaStream_t stream);

/* Synchronizes `stream`, then reads and clears the current device's status
 * word: WISE_OK, WISE_ERR_BAD_SUPPORT or WISE_ERR_TIMEOUT (the latter wins
 * when both were recorded), or WISE_ERR_CUDA if the synchronization failed. */
int wise_get_status(cudaStream_t stream);

/* Sets the time limit of each internal wait of the attention kernels
 * (wise_full_attn_accumulate, its _noalloc variant, wise_sparse_attn and
 * wise_freeze_a_attn) for every later launch in this process; ns == 0
 * restores the default of 2 s.  A wait that runs out makes the kernel stop
 * issuing work, let the work already in flight finish, and record
 * WISE_ERR_TIMEOUT for wise_get_status(); the outputs of that launch are then
 * incomplete.  The waits of that unwinding keep the 2 s limit.  Process-wide
 * (not per device or stream); always returns WISE_OK.  The paper has no
 * counterpart: this is the failure-detection control of the kernels. */
int wise_set_wait_limit_ns(unsigned long long ns);

/* Static description of a status code. */
const char* wise_status_string(int status);

/* Library version, major * 10000 + minor * 100 + patch. */
int wise_version(void);

#ifdef __cplusplus
}
#endif

#endif /* WISE_H_ */
