/*
 * Slot-attention oracle: plain, slow, fp64 CPU code.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may call this file;
 * only the tests, the smoke check and the benchmark's CPU-baseline leg do.
 * It shares no code, header or constant with the CUDA library.
 *
 * What it computes (Zarya, Sec. 5.2 "Slotted speculative decoding", steps 3
 * and 6, with the KV-reuse argument of Sec. 5.1 and Sec. 3.1):
 *   a block of S_b slots x L_b tokens (R_b = S_b * L_b query rows) of
 *   sequence b, placed after the committed prefix of P_b = cache_lens[b]
 *   tokens by the reordering step, attends over the cached prefix keys plus
 *   the block's own keys (staged at cache positions P_b .. P_b + R_b - 1):
 *
 *     sigma_c = scale * sum_d q[r, h, d] * k[c, h / g, d]      (g = Hq / Hkv)
 *     out[r, h, :] = sum_{c visible} exp(sigma_c - m) v[c, h / g, :]
 *                    / sum_{c visible} exp(sigma_c - m),  m = max sigma_c
 *
 *   visible(c) for row r:
 *     mode 0 (block-bidirectional, draft / diffusion selection, step 3):
 *       c < P_b + R_b
 *     mode 1 (slot-causal, verification / AR infilling, step 6):
 *       c < P_b + r + 1   (causal over the reordered, flattened sequence)
 *     mode 2 (slot-independent verification: each selected slot verified on
 *       its own, step 6 run for several slots in one pass), for row
 *       r = s * L_b + j (slot s, offset j):
 *       c < P_b  or  P_b + s * L_b <= c <= P_b + r
 *
 * Every value is read exactly (bf16 / fp32 -> fp64 is exact) and every sum is
 * taken in fp64 in key order. No tiling, no online softmax, no splitting.
 *
 * Cache layouts (token c of sequence b, kv head j, element d):
 *   contiguous (page_size == 0): k[((b * capacity + c) * Hkv + j) * D + d]
 *   paged      (page_size  > 0): page p = page_table[b * max_pages + c / page_size],
 *                                k[((p * page_size + c % page_size) * Hkv + j) * D + d]
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* element types of the input arrays */
enum { OR_F64 = 0, OR_F32 = 1, OR_BF16 = 2 };

static double load_elem(const void* base, int64_t i, int dtype) {
  if (dtype == OR_F64) return ((const double*)base)[i];
  if (dtype == OR_F32) return (double)((const float*)base)[i];
  /* bf16: the upper 16 bits of an IEEE binary32 */
  uint32_t bits = ((uint32_t)((const uint16_t*)base)[i]) << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

typedef struct {
  const void* q;
  const void* k;
  const void* v;
  int dtype;
  const int32_t* cache_lens;
  const int32_t* page_table;
  int32_t max_pages;
  int32_t page_size;
  int32_t capacity;
  const int32_t* n_slots;
  const int32_t* slot_len;
  const int32_t* mask_mode;
  const int64_t* q_row_offsets;
  int32_t B, Hq, Hkv, D;
  double scale;
} or_problem;

/* flat element index of (token c, kv head j, element 0) of sequence b; -1 if
 * the page table entry is out of range */
static int64_t kv_index(const or_problem* p, int b, int64_t c, int j, int64_t n_pages) {
  int64_t tok;
  if (p->page_size == 0) {
    tok = (int64_t)b * p->capacity + c;
  } else {
    int64_t page = p->page_table[(int64_t)b * p->max_pages + c / p->page_size];
    if (page < 0 || (n_pages >= 0 && page >= n_pages)) return -1;
    tok = page * p->page_size + c % p->page_size;
  }
  return (tok * p->Hkv + j) * p->D;
}

/* One output row out[0..D) for (sequence b, query head h, block row r).
 * Returns 0 on success, -1 on an invalid argument. */
static int attend_one(const or_problem* p, int b, int h, int r, int64_t n_pages, double* out,
                      double* sigma /* scratch, >= P_b + R_b */) {
  const int g = p->Hq / p->Hkv;
  const int j = h / g;
  const int64_t P = p->cache_lens[b];
  const int64_t R = (int64_t)p->n_slots[b] * p->slot_len[b];
  if (r < 0 || r >= R) return -1;
  const int mode = p->mask_mode[b];
  if (mode < 0 || mode > 2) return -1;
  /* keys beyond the last visible one are never read */
  const int64_t n_vis = (mode == 0) ? P + R : P + r + 1;
  /* mode 2 also hides the block rows of the earlier slots: [P, P + s * L) */
  const int64_t L = p->slot_len[b];
  const int64_t hide_lo = P, hide_hi = (mode == 2) ? P + (r / L) * L : P;

  const int64_t qbase = ((p->q_row_offsets[b] + r) * p->Hq + h) * (int64_t)p->D;
  double m = -INFINITY;
  for (int64_t c = 0; c < n_vis; ++c) {
    if (c >= hide_lo && c < hide_hi) continue;
    const int64_t kb = kv_index(p, b, c, j, n_pages);
    if (kb < 0) return -1;
    double dot = 0.0;
    for (int d = 0; d < p->D; ++d)
      dot += load_elem(p->q, qbase + d, p->dtype) * load_elem(p->k, kb + d, p->dtype);
    sigma[c] = p->scale * dot;
    if (sigma[c] > m) m = sigma[c];
  }
  double denom = 0.0;
  for (int d = 0; d < p->D; ++d) out[d] = 0.0;
  for (int64_t c = 0; c < n_vis; ++c) {
    if (c >= hide_lo && c < hide_hi) continue;
    const double w = exp(sigma[c] - m);
    denom += w;
    const int64_t vb = kv_index(p, b, c, j, n_pages);
    for (int d = 0; d < p->D; ++d) out[d] += w * load_elem(p->v, vb + d, p->dtype);
  }
  for (int d = 0; d < p->D; ++d) out[d] /= denom;
  return 0;
}

static int64_t max_keys(const or_problem* p) {
  int64_t mx = 1;
  for (int b = 0; b < p->B; ++b) {
    int64_t n = (int64_t)p->cache_lens[b] + (int64_t)p->n_slots[b] * p->slot_len[b];
    if (n > mx) mx = n;
  }
  return mx;
}

/*
 * Full output: out[(q_row_offsets[b] + r) * Hq + h][D] for every b, h and
 * r < R_b (fp64). Rows of q beyond q_row_offsets[B] are not touched.
 * Returns 0, or -1 if an argument is invalid (bad mode, page id, head count).
 */
int oracle_slot_attn(const void* q, const void* k_cache, const void* v_cache, int dtype,
                     const int32_t* cache_lens, const int32_t* page_table, int32_t max_pages,
                     int32_t page_size, int32_t capacity, int64_t n_pages,
                     const int32_t* n_slots, const int32_t* slot_len, const int32_t* mask_mode,
                     const int64_t* q_row_offsets, int32_t B, int32_t Hq, int32_t Hkv,
                     int32_t D, double scale, double* out, int32_t n_threads) {
  if (B <= 0 || Hkv <= 0 || Hq <= 0 || Hq % Hkv != 0 || D <= 0) return -1;
  or_problem p = {q, k_cache, v_cache, dtype, cache_lens, page_table, max_pages, page_size,
                  capacity, n_slots, slot_len, mask_mode, q_row_offsets, B, Hq, Hkv, D, scale};
  const int64_t mk = max_keys(&p);
  int64_t n_units = (int64_t)B * Hq;
  int failed = 0;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel reduction(| : failed)
#endif
  {
    double* sigma = (double*)malloc(sizeof(double) * (size_t)mk);
    if (!sigma) failed = 1;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
    for (int64_t u = 0; u < n_units; ++u) {
      if (!sigma) continue;
      const int b = (int)(u / Hq), h = (int)(u % Hq);
      const int64_t R = (int64_t)n_slots[b] * slot_len[b];
      for (int64_t r = 0; r < R; ++r) {
        double* o = out + ((q_row_offsets[b] + r) * Hq + h) * (int64_t)D;
        if (attend_one(&p, b, h, (int)r, n_pages, o, sigma) != 0) failed = 1;
      }
    }
    free(sigma);
  }
  (void)n_threads;
  return failed ? -1 : 0;
}

/*
 * Selected outputs only: for i < n_sel, sel[3i..3i+2] = (b, h, r) and
 * out[i][D] receives that row. Used to check full-size launches on samples.
 */
int oracle_slot_attn_rows(const void* q, const void* k_cache, const void* v_cache, int dtype,
                          const int32_t* cache_lens, const int32_t* page_table,
                          int32_t max_pages, int32_t page_size, int32_t capacity,
                          int64_t n_pages, const int32_t* n_slots, const int32_t* slot_len,
                          const int32_t* mask_mode, const int64_t* q_row_offsets, int32_t B,
                          int32_t Hq, int32_t Hkv, int32_t D, double scale, const int64_t* sel,
                          int64_t n_sel, double* out, int32_t n_threads) {
  if (B <= 0 || Hkv <= 0 || Hq <= 0 || Hq % Hkv != 0 || D <= 0) return -1;
  or_problem p = {q, k_cache, v_cache, dtype, cache_lens, page_table, max_pages, page_size,
                  capacity, n_slots, slot_len, mask_mode, q_row_offsets, B, Hq, Hkv, D, scale};
  const int64_t mk = max_keys(&p);
  int failed = 0;
#ifdef _OPENMP
  if (n_threads > 0) omp_set_num_threads(n_threads);
#pragma omp parallel reduction(| : failed)
#endif
  {
    double* sigma = (double*)malloc(sizeof(double) * (size_t)mk);
    if (!sigma) failed = 1;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
    for (int64_t i = 0; i < n_sel; ++i) {
      if (!sigma) continue;
      const int64_t b = sel[3 * i], h = sel[3 * i + 1], r = sel[3 * i + 2];
      if (b < 0 || b >= B || h < 0 || h >= Hq) { failed = 1; continue; }
      if (attend_one(&p, (int)b, (int)h, (int)r, n_pages, out + i * (int64_t)D, sigma) != 0)
        failed = 1;
    }
    free(sigma);
  }
  (void)n_threads;
  return failed ? -1 : 0;
}

/* Number of OpenMP threads a parallel region would use (1 without OpenMP). */
int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
