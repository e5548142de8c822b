/*
 * fp64 CPU oracle for the WISE attention hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, plainly written checker
 * the CUDA path is compared against.  Only the tests, the smoke check and the
 * benchmark's CPU-baseline leg may build, load or call it; the library under
 * paper_2609_27373_gb300/ never does, and shares no code with it.
 *
 * What it computes, each function following one passage of the paper
 * ("Attention Routing Stabilizes Early: Working-Set Inference for
 * Recurrent-Depth Language Models"):
 *
 *   wo_full_attention    Eq. 2  A = softmax(QK^T/sqrt(d_h) + M), O = AV, with
 *                               M the causal mask, and Eq. 5 block mass
 *                               r_qb = (1/|I_q|) sum_{i in I_q} sum_{j in I_b} A_ij
 *   wo_select_support    Eq. 6  block support selection, in the single-pass
 *                               form used by the benchmark workloads (sink and
 *                               local blocks forced, then top-k or cumulative
 *                               mass coverage over the accumulated masses)
 *   wo_sparse_attention  Eqs. 7-8  attention restricted to the block support:
 *                               R_ij = 0 if b(j) in B_q(i) else -inf
 *
 * Inputs are bf16 bit patterns (uint16), widened exactly to double; all
 * arithmetic is double.  Selection runs on fp32 block masses with exact
 * integer fixed-point rules so that any two correct implementations agree
 * bit for bit:
 *   u(x)   = floor(min(x, 4096) * 2^32) for x > 0, else 0 (NaN -> 0)
 *   U[kb]  = sum of u over the query heads of the kv-head group
 *   rank   = (U descending, kb ascending)  -- ties go to the lowest block
 *   eta16  = floor(eta * 65536 + 0.5); coverage holds once
 *            cum * 65536 >= eta16 * T, with T = sum of U over kb in [0, q]
 * Parity of the selection is therefore exact; the attention values are only
 * as close to the GPU as bf16 inputs with fp32 accumulation allow.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
  int batch, seqlen, n_heads, n_kv_heads, head_dim, block;
  double scale; /* <= 0 selects 1/sqrt(head_dim) (Eq. 2) */
} wo_shape;

typedef struct {
  int n_sink;   /* blocks 0 .. n_sink-1 are always kept */
  int n_local;  /* blocks q-n_local+1 .. q are always kept (1 = diagonal) */
  int mode;     /* 0 = top-k, 1 = cumulative-mass coverage */
  int topk;     /* top-k: number of ranked blocks added to the forced ones */
  float eta;    /* coverage: mass threshold in [0, 1] */
  int cap;      /* maximum support size, forced blocks included */
} wo_select;

static double bf16_value(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static double shape_scale(const wo_shape* s) {
  return s->scale > 0.0 ? s->scale : 1.0 / sqrt((double)s->head_dim);
}

static int shape_ok(const wo_shape* s) {
  if (s->batch < 0 || s->seqlen < 0 || s->n_heads <= 0 || s->n_kv_heads <= 0 || s->head_dim <= 0 ||
      s->block <= 0)
    return 0;
  if (s->n_heads % s->n_kv_heads) return 0;
  if (s->seqlen % s->block) return 0;
  return 1;
}

int wo_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

void wo_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* One query row under Eq. 2 / Eq. 8: the logits of the admissible keys,
 * their softmax, the output row, and (if mass_row != NULL) the row's
 * contribution A_ij / |I_q| to r_{q b(j)} (Eq. 5). keep[j] != 0 marks the
 * admissible keys j (j <= i always). */
static void attend_row(const wo_shape* s, const uint16_t* q_row, const uint16_t* Kh, const uint16_t* Vh,
                       int i, const unsigned char* keep_block, double* logit, double* o_row,
                       double* mass_row) {
  const int D = s->head_dim, B = s->block;
  const double scale = shape_scale(s);
  double mx = -INFINITY;
  int any = 0;
  for (int j = 0; j <= i; ++j) {
    if (keep_block && !keep_block[j / B]) continue;
    double dot = 0.0;
    for (int k = 0; k < D; ++k) dot += bf16_value(q_row[k]) * bf16_value(Kh[(size_t)j * D + k]);
    logit[j] = scale * dot;
    if (logit[j] > mx) mx = logit[j];
    any = 1;
  }
  for (int k = 0; k < D; ++k) o_row[k] = 0.0;
  if (!any) return; /* no admissible key: the output row is defined as 0 */
  double z = 0.0;
  for (int j = 0; j <= i; ++j) {
    if (keep_block && !keep_block[j / B]) continue;
    logit[j] = exp(logit[j] - mx);
    z += logit[j];
  }
  for (int j = 0; j <= i; ++j) {
    if (keep_block && !keep_block[j / B]) continue;
    const double a = logit[j] / z; /* A_ij */
    for (int k = 0; k < D; ++k) o_row[k] += a * bf16_value(Vh[(size_t)j * D + k]);
    if (mass_row) mass_row[j / B] += a / (double)B;
  }
}

/* Decode unit u of the (b, h, q) list; units == NULL means all units in
 * (b, h, q) order. */
static void unit_at(const wo_shape* s, const int32_t* units, long u, int* b, int* h, int* q) {
  if (units) {
    *b = units[3 * u];
    *h = units[3 * u + 1];
    *q = units[3 * u + 2];
  } else {
    const int nq = s->seqlen / s->block;
    *q = (int)(u % nq);
    *h = (int)((u / nq) % s->n_heads);
    *b = (int)(u / ((long)nq * s->n_heads));
  }
}

/* Eq. 2 with the causal mask, and Eq. 5.
 * Q [batch, n_heads, L, D], K/V [batch, n_kv_heads, L, D] as bf16 bits.
 * With units == NULL every query block is computed and O is
 * [batch, n_heads, L, D], mass [batch, n_heads, nQB, nKB] (double, mass may
 * be NULL).  With a list of n_units (b, h, q) triples only those blocks are
 * computed and the outputs are packed per unit: O [n_units, block, D],
 * mass [n_units, nKB].  Returns 0, or -1 on a bad shape or unit. */
int wo_full_attention(const wo_shape* s, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                      long n_units, const int32_t* units, double* O, double* mass) {
  if (!shape_ok(s)) return -1;
  const int L = s->seqlen, D = s->head_dim, B = s->block, nb = L / B, grp = s->n_heads / s->n_kv_heads;
  const long total = units ? n_units : (long)s->batch * s->n_heads * nb;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (long u = 0; u < total; ++u) {
    int b, h, q;
    unit_at(s, units, u, &b, &h, &q);
    if (b < 0 || b >= s->batch || h < 0 || h >= s->n_heads || q < 0 || q >= nb) {
      bad = 1;
      continue;
    }
    const int g = h / grp;
    const uint16_t* Qh = Q + ((size_t)b * s->n_heads + h) * L * D;
    const uint16_t* Kh = K + ((size_t)b * s->n_kv_heads + g) * L * D;
    const uint16_t* Vh = V + ((size_t)b * s->n_kv_heads + g) * L * D;
    double* logit = (double*)malloc(sizeof(double) * (size_t)L);
    double* mass_row = !mass ? NULL : units ? mass + (size_t)u * nb : mass + (((size_t)b * s->n_heads + h) * nb + q) * nb;
    double* o_blk = units ? O + (size_t)u * B * D : O + (((size_t)b * s->n_heads + h) * L + (size_t)q * B) * D;
    if (mass_row)
      for (int kb = 0; kb < nb; ++kb) mass_row[kb] = 0.0;
    for (int i = q * B; i < (q + 1) * B; ++i)
      attend_row(s, Qh + (size_t)i * D, Kh, Vh, i, NULL, logit, o_blk + (size_t)(i - q * B) * D, mass_row);
    free(logit);
  }
  return bad ? -1 : 0;
}

/* Eqs. 7-8: attention restricted to the block support of each query block.
 * idx [batch, n_kv_heads, nQB, cap] (ascending block ids, padded with -1),
 * counts [batch, n_kv_heads, nQB]; a query head uses its kv-head group's
 * support.  O is laid out as in wo_full_attention.  Returns -1 if a shape is bad, a count exceeds cap, or a listed
 * block lies outside [0, nKB). */
int wo_sparse_attention(const wo_shape* s, const uint16_t* Q, const uint16_t* K, const uint16_t* V,
                        const int32_t* idx, const int32_t* counts, int cap, long n_units,
                        const int32_t* units, double* O) {
  if (!shape_ok(s) || cap <= 0) return -1;
  const int L = s->seqlen, D = s->head_dim, B = s->block, nb = L / B, grp = s->n_heads / s->n_kv_heads;
  const long total = units ? n_units : (long)s->batch * s->n_heads * nb;
  int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
  for (long u = 0; u < total; ++u) {
    int b, h, q;
    unit_at(s, units, u, &b, &h, &q);
    if (b < 0 || b >= s->batch || h < 0 || h >= s->n_heads || q < 0 || q >= nb) {
      bad = 1;
      continue;
    }
    const int g = h / grp;
    const size_t row = ((size_t)b * s->n_kv_heads + g) * nb + q;
    const int n = counts[row];
    unsigned char* keep = (unsigned char*)calloc((size_t)nb, 1);
    if (n < 0 || n > cap) bad = 1;
    for (int t = 0; t < n && t < cap; ++t) {
      const int kb = idx[row * cap + t];
      if (kb < 0 || kb >= nb)
        bad = 1;
      else
        keep[kb] = 1;
    }
    const uint16_t* Qh = Q + ((size_t)b * s->n_heads + h) * L * D;
    const uint16_t* Kh = K + ((size_t)b * s->n_kv_heads + g) * L * D;
    const uint16_t* Vh = V + ((size_t)b * s->n_kv_heads + g) * L * D;
    double* logit = (double*)malloc(sizeof(double) * (size_t)L);
    double* o_blk = units ? O + (size_t)u * B * D : O + (((size_t)b * s->n_heads + h) * L + (size_t)q * B) * D;
    for (int i = q * B; i < (q + 1) * B; ++i)
      attend_row(s, Qh + (size_t)i * D, Kh, Vh, i, keep, logit, o_blk + (size_t)(i - q * B) * D, NULL);
    free(logit);
    free(keep);
  }
  return bad ? -1 : 0;
}

/* Fixed-point mass u(x) = floor(min(x, 4096) * 2^32), 0 unless x > 0. */
static uint64_t mass_units(float x) {
  if (!(x > 0.0f)) return 0;
  if (x > 4096.0f) x = 4096.0f;
  return (uint64_t)floor((double)x * 4294967296.0);
}

typedef struct {
  uint64_t U;
  int kb;
} ranked_t;

/* Rank order: larger pooled mass first, then the lower block index. */
static int rank_cmp(const void* a, const void* b) {
  const ranked_t* x = (const ranked_t*)a;
  const ranked_t* y = (const ranked_t*)b;
  if (x->U != y->U) return x->U > y->U ? -1 : 1;
  return (x->kb > y->kb) - (x->kb < y->kb);
}

static int int_cmp(const void* a, const void* b) {
  const int x = *(const int*)a, y = *(const int*)b;
  return (x > y) - (x < y);
}

/* Support selection (Eq. 6, single-pass form over accumulated masses).
 * blockmass [batch, n_heads, nQB, nKB] fp32; only entries kb <= q are read.
 * idx [batch, n_kv_heads, nQB, cap] int32 (ascending, padded with -1),
 * counts [batch, n_kv_heads, nQB].  Returns -1 on invalid arguments. */
int wo_select_support(const wo_shape* s, const wo_select* sel, const float* blockmass, int32_t* idx,
                      int32_t* counts) {
  if (!shape_ok(s)) return -1;
  if (sel->n_sink < 0 || sel->n_local < 1 || sel->cap < sel->n_sink + sel->n_local) return -1;
  if (sel->mode == 0 && sel->topk < 0) return -1;
  if (sel->mode == 1 && !(sel->eta >= 0.0f && sel->eta <= 1.0f)) return -1;
  if (sel->mode != 0 && sel->mode != 1) return -1;
  const int nb = s->seqlen / s->block, grp = s->n_heads / s->n_kv_heads, cap = sel->cap;
  const uint64_t eta16 = (uint64_t)floor((double)sel->eta * 65536.0 + 0.5);
  const long rows = (long)s->batch * s->n_kv_heads * nb;
#pragma omp parallel for schedule(dynamic, 16)
  for (long r = 0; r < rows; ++r) {
    const int q = (int)(r % nb);
    const int g = (int)((r / nb) % s->n_kv_heads);
    const int b = (int)(r / ((long)nb * s->n_kv_heads));
    uint64_t* U = (uint64_t*)calloc((size_t)nb, sizeof(uint64_t));
    unsigned char* forced = (unsigned char*)calloc((size_t)nb, 1);
    ranked_t* cand = (ranked_t*)malloc(sizeof(ranked_t) * (size_t)nb);
    int* chosen = (int*)malloc(sizeof(int) * (size_t)nb);
    for (int h = g * grp; h < (g + 1) * grp; ++h) {
      const float* m = blockmass + (((size_t)b * s->n_heads + h) * nb + q) * nb;
      for (int kb = 0; kb <= q; ++kb) U[kb] += mass_units(m[kb]);
    }
    int n = 0;
    for (int kb = 0; kb <= q; ++kb) {
      if (kb < sel->n_sink || kb > q - sel->n_local) {
        forced[kb] = 1;
        chosen[n++] = kb;
      }
    }
    int nc = 0;
    for (int kb = 0; kb <= q; ++kb)
      if (!forced[kb]) {
        cand[nc].U = U[kb];
        cand[nc].kb = kb;
        ++nc;
      }
    qsort(cand, (size_t)nc, sizeof(ranked_t), rank_cmp);
    if (sel->mode == 0) {
      for (int t = 0; t < nc && t < sel->topk && n < cap; ++t) chosen[n++] = cand[t].kb;
    } else {
      uint64_t T = 0, cum = 0;
      for (int kb = 0; kb <= q; ++kb) T += U[kb];
      for (int t = 0; t < n; ++t) cum += U[chosen[t]];
      int t = 0;
      while ((unsigned __int128)cum * 65536u < (unsigned __int128)eta16 * T && n < cap && t < nc) {
        cum += cand[t].U;
        chosen[n++] = cand[t].kb;
        ++t;
      }
    }
    qsort(chosen, (size_t)n, sizeof(int), int_cmp);
    for (int t = 0; t < cap; ++t) idx[r * cap + t] = t < n ? chosen[t] : -1;
    counts[r] = n;
    free(U);
    free(forced);
    free(cand);
    free(chosen);
  }
  return 0;
}
