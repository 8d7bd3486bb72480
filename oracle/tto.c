/*
 * tto.c -- CPU oracle of the TokenTiming verification path (arXiv 2510.15545).
 *
 * TEST INFRASTRUCTURE: the plain, slow, obviously-correct definition that the
 * CUDA path is checked against. Only the tests, the smoke check and the
 * benchmark's CPU legs may load it. It shares nothing with the CUDA library.
 *
 * Readings of the paper taken here (each one is listed with its reason in the
 * design notes of the repository):
 *  - p is the target distribution, q the draft one, accept while
 *    u < min(1, p/q) (Alg. 4 naming; §3 and Alg. 2 swap the letters).
 *  - Band: |i - j| <= w_eff with w_eff = max(w, |k - m|), so (k, m) is always
 *    reachable; w < 0 means no band (§4.1 band, Alg. 1).
 *  - Backtrack ties: prefer (i-1, j-1), then (i-1, j), then (i, j-1).
 *  - Token distance is Levenshtein over the tokens' UTF-8 bytes (App. H, and
 *    the byte-level resolution of the fragmented-tokenization study).
 *  - Transfer: target position j takes the draft token with the largest i
 *    aligned to it (terminal rule for many-to-one, copy rule for one-to-many,
 *    App. A.2); its probability is the one-hot probability of that sampled
 *    draft token (Limitations).
 *  - After a rejection at j the next token is drawn from the normalised
 *    residual max(0, p_j - q_j) (Alg. 4); with the one-hot q this is p_j with
 *    the rejected token's mass reduced to max(0, p_j(t) - q_hat_j).
 *  - Uniforms: Philox4x64-10, counter (position, stream, request, 0), key
 *    (seed, 0), u = top 24 bits * 2^-24; stream 0 = accept, 1 = resample.
 */
#include "tto.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

#define ST_ID_RANGE 1
#define ST_TOO_LONG 2
#define ST_EMPTY 4
#define ST_BAD_OFFSETS 8
#define ST_NO_MATCH 128
#define ST_INCONSISTENT 256
#define MAX_K 256
#define MAX_M 512
#define MAX_TOKEN_BYTES 256
#define BOUNDARY_EPS 1e-6

/* ------------------------------------------------------------------ App. H */

int32_t tto_lev(const uint8_t* s, int32_t ns, const uint8_t* t, int32_t nt) {
  /* D(i,0) = i, D(0,j) = j; D(i,j) = min(D(i-1,j)+1, D(i,j-1)+1,
   * D(i-1,j-1) + [s_i != t_j]); the distance is D(ns, nt). */
  int32_t* D = (int32_t*)malloc(sizeof(int32_t) * (size_t)(ns + 1) * (size_t)(nt + 1));
  int32_t W = nt + 1;
  for (int32_t i = 0; i <= ns; ++i) D[i * W] = i;
  for (int32_t j = 0; j <= nt; ++j) D[j] = j;
  for (int32_t i = 1; i <= ns; ++i) {
    for (int32_t j = 1; j <= nt; ++j) {
      int32_t del = D[(i - 1) * W + j] + 1;
      int32_t ins = D[i * W + (j - 1)] + 1;
      int32_t sub = D[(i - 1) * W + (j - 1)] + (s[i - 1] == t[j - 1] ? 0 : 1);
      int32_t best = del < ins ? del : ins;
      D[i * W + j] = sub < best ? sub : best;
    }
  }
  int32_t r = D[ns * W + nt];
  free(D);
  return r;
}

/* ------------------------------------------------------------------ Alg. 1 */

#define DTW_INF ((int64_t)1 << 60)

int64_t tto_dtw(int32_t k, int32_t m, const int32_t* d, int32_t w,
                int32_t* path, int32_t* path_len) {
  *path_len = 0;
  if (k <= 0 || m <= 0) return -1;
  int64_t band;
  if (w < 0) {
    band = (int64_t)k + m; /* no band */
  } else {
    int64_t gap = k > m ? k - m : m - k;
    band = w > gap ? w : gap;
  }
  int64_t W = m + 1;
  int64_t* C = (int64_t*)malloc(sizeof(int64_t) * (size_t)(k + 1) * (size_t)W);
  for (int64_t x = 0; x < (int64_t)(k + 1) * W; ++x) C[x] = DTW_INF;
  C[0] = 0; /* C_{0,0} = 0, every other border cell is infinite */
  for (int32_t i = 1; i <= k; ++i) {
    int64_t jlo = i - band > 1 ? i - band : 1;
    int64_t jhi = i + band < m ? i + band : m;
    for (int64_t j = jlo; j <= jhi; ++j) {
      int64_t up = C[(i - 1) * W + j];
      int64_t left = C[i * W + (j - 1)];
      int64_t diag = C[(i - 1) * W + (j - 1)];
      int64_t best = up < left ? up : left;
      best = diag < best ? diag : best;
      C[i * W + j] = best >= DTW_INF ? DTW_INF : best + d[(int64_t)(i - 1) * m + (j - 1)];
    }
  }
  int64_t cstar = C[(int64_t)k * W + m];
  if (cstar >= DTW_INF) {
    free(C);
    return -1;
  }
  /* Backtrack from (k, m) to (0, 0), collecting cells in reverse order. */
  int32_t* rev = (int32_t*)malloc(sizeof(int32_t) * 2 * (size_t)(k + m));
  int32_t L = 0;
  int64_t i = k, j = m;
  while (i != 0 || j != 0) {
    rev[2 * L] = (int32_t)i;
    rev[2 * L + 1] = (int32_t)j;
    ++L;
    /* candidates in preference order: diagonal, up, left */
    int64_t bi = i - 1, bj = j - 1;
    int64_t bc = (bi >= 0 && bj >= 0) ? C[bi * W + bj] : DTW_INF;
    int64_t cu = (i - 1 >= 0) ? C[(i - 1) * W + j] : DTW_INF;
    if (cu < bc) { bi = i - 1; bj = j; bc = cu; }
    int64_t cl = (j - 1 >= 0) ? C[i * W + (j - 1)] : DTW_INF;
    if (cl < bc) { bi = i; bj = j - 1; bc = cl; }
    i = bi;
    j = bj;
  }
  for (int32_t x = 0; x < L; ++x) { /* forward order, 0-based indices */
    path[2 * x] = rev[2 * (L - 1 - x)] - 1;
    path[2 * x + 1] = rev[2 * (L - 1 - x) + 1] - 1;
  }
  *path_len = L;
  free(rev);
  free(C);
  return cstar;
}

/* ------------------------------------------------ Philox (Salmon et al. 2011) */

static void mulhilo64(uint64_t a, uint64_t b, uint64_t* hi, uint64_t* lo) {
  unsigned __int128 p = (unsigned __int128)a * (unsigned __int128)b;
  *hi = (uint64_t)(p >> 64);
  *lo = (uint64_t)p;
}

void tto_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2], uint64_t out[4]) {
  const uint64_t M0 = 0xD2E7470EE14C6C93ULL, M1 = 0xCA5A826395121157ULL;
  const uint64_t W0 = 0x9E3779B97F4A7C15ULL, W1 = 0xBB67AE8584CAA73BULL;
  uint64_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint64_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    uint64_t hi0, lo0, hi1, lo1;
    mulhilo64(M0, c0, &hi0, &lo0);
    mulhilo64(M1, c2, &hi1, &lo1);
    uint64_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    k0 += W0;
    k1 += W1;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

double tto_uniform(uint64_t seed, uint64_t pos, uint64_t stream, uint64_t request) {
  uint64_t ctr[4] = {pos, stream, request, 0}, key[2] = {seed, 0}, out[4];
  tto_philox4x64_10(ctr, key, out);
  return (double)(out[0] >> 40) * (1.0 / 16777216.0);
}

/* ------------------------------------------------------------------ softmax */

static double load_logit(const void* row, int32_t dtype, int64_t x) {
  if (dtype == 0) return (double)((const float*)row)[x];
  /* bf16: the upper 16 bits of an IEEE binary32 */
  uint32_t bits = (uint32_t)((const uint16_t*)row)[x] << 16;
  float f;
  memcpy(&f, &bits, sizeof f);
  return (double)f;
}

static const void* row_ptr(const void* base, int32_t dtype, int64_t stride, int64_t r) {
  size_t elem = dtype == 0 ? 4 : 2;
  return (const char*)base + (size_t)r * (size_t)stride * elem;
}

double tto_logsumexp(const void* row, int32_t dtype, int64_t V, double T) {
  double mx = -INFINITY;
  for (int64_t x = 0; x < V; ++x) {
    double z = load_logit(row, dtype, x) / T;
    if (z > mx) mx = z;
  }
  double s = 0.0;
  for (int64_t x = 0; x < V; ++x) s += exp(load_logit(row, dtype, x) / T - mx);
  return mx + log(s);
}

void tto_softmax(const void* row, int32_t dtype, int64_t V, double T, double* p) {
  double mx = -INFINITY;
  for (int64_t x = 0; x < V; ++x) {
    double z = load_logit(row, dtype, x) / T;
    if (z > mx) mx = z;
  }
  double s = 0.0;
  for (int64_t x = 0; x < V; ++x) {
    p[x] = exp(load_logit(row, dtype, x) / T - mx);
    s += p[x];
  }
  for (int64_t x = 0; x < V; ++x) p[x] /= s;
}

/* ------------------------------------------------------------ batched align */

/* ------------------------------------------------------- sampling filters */

/* The generation filters of the paper's hyperparameter table, in the usual
 * order: temperature, then top-k (keep the k largest logits; among equal
 * logits the smaller column first), then top-p (after renormalising, keep
 * tokens in decreasing probability while the mass before a token is below
 * top_p, so the kept set is the smallest prefix reaching top_p). top_k <= 0 or
 * top_k >= V: no top-k; top_p <= 0 or >= 1: no top-p. Writes the filtered
 * distribution over all V columns (zeros outside the kept set) and returns the
 * natural log of the kept set's normaliser sum exp(z/T). *boundary gets bit 4
 * when the mass before some token lies within 1e-6 of top_p. */
static const void* g_sort_row; /* the row the comparator reads (single-threaded) */
static int32_t g_sort_dtype;
static double sort_val(int64_t x) { return load_logit(g_sort_row, g_sort_dtype, x); }
static int cmp_desc_logit(const void* pa, const void* pb) {
  int64_t a = *(const int64_t*)pa, b = *(const int64_t*)pb;
  double va = sort_val(a), vb = sort_val(b);
  if (va > vb) return -1;
  if (va < vb) return 1;
  return a < b ? -1 : (a > b ? 1 : 0);
}

double tto_filtered_probs(const void* row, int32_t dtype, int64_t V, double T, int32_t top_k,
                          double top_p, double* p, int32_t* boundary) {
  int64_t* order = (int64_t*)malloc(sizeof(int64_t) * (size_t)V);
  for (int64_t x = 0; x < V; ++x) order[x] = x;
  g_sort_row = row;
  g_sort_dtype = dtype;
  qsort(order, (size_t)V, sizeof(int64_t), cmp_desc_logit);
  int64_t K = (top_k <= 0 || top_k >= V) ? V : top_k;
  /* softmax over the top-K (the maximum is the first) */
  double mx = load_logit(row, dtype, order[0]) / T, sum = 0.0;
  for (int64_t i = 0; i < K; ++i) sum += exp(load_logit(row, dtype, order[i]) / T - mx);
  int64_t keep = K;
  if (top_p > 0.0 && top_p < 1.0) {
    double before = 0.0;
    keep = 0;
    while (keep < K) {
      if (fabs(before - top_p) < 1e-6 && boundary) *boundary |= 4;
      if (!(before < top_p)) break;
      before += exp(load_logit(row, dtype, order[keep]) / T - mx) / sum;
      ++keep;
    }
  }
  double kept = 0.0;
  for (int64_t i = 0; i < keep; ++i) kept += exp(load_logit(row, dtype, order[i]) / T - mx);
  for (int64_t x = 0; x < V; ++x) p[x] = 0.0;
  for (int64_t i = 0; i < keep; ++i)
    p[order[i]] = exp(load_logit(row, dtype, order[i]) / T - mx) / kept;
  free(order);
  return mx + log(kept);
}

static int32_t offsets_ok(const int32_t* off, int32_t b) {
  return off[b] >= 0 && off[b + 1] >= off[b];
}

/* ------------------------------------------------------ repetition penalty */

/* The repetition penalty of the generation hyperparameters (App. F; the
 * Hugging Face default the paper says it keeps): every column of the row's
 * penalized set -- the request's history and the sequence tokens before the
 * row's position -- has its logit z replaced by z * theta when z < 0 and by
 * z / theta otherwise, once however often the column occurs, in fp32
 * arithmetic (the logits' own type); temperature and the filters then act on
 * the penalized row. Returns the row to use: `row` itself when there is no
 * penalty, else `buf` (V floats) holding the penalized copy. */
static const void* penalized_row(const void* row, int32_t dtype, int64_t V,
                                 const tto_penalty* pen, int32_t b, const int32_t* seq,
                                 int32_t n_seq, float* buf, uint8_t* mark, int32_t* out_dtype) {
  if (!pen || pen->theta == 1.0f) {
    *out_dtype = dtype;
    return row;
  }
  for (int64_t x = 0; x < V; ++x) {
    buf[x] = (float)load_logit(row, dtype, x);
    mark[x] = 0;
  }
  if (pen->hist_off)
    for (int32_t h = pen->hist_off[b]; h < pen->hist_off[b + 1]; ++h) {
      const int32_t c = pen->hist_cols[h];
      if (c >= 0 && c < V) mark[c] = 1;
    }
  for (int32_t i = 0; i < n_seq; ++i)
    if (seq[i] >= 0 && seq[i] < V) mark[seq[i]] = 1;
  const float theta = pen->theta;
  for (int64_t x = 0; x < V; ++x)
    if (mark[x]) buf[x] = buf[x] < 0.0f ? buf[x] * theta : buf[x] / theta;
  *out_dtype = 0;
  return buf;
}

/* Status of a request's history under a penalty: its CSR range and columns. */
static int32_t history_status(const tto_penalty* pen, int32_t b, int64_t V) {
  if (!pen || pen->theta == 1.0f || !pen->hist_off) return 0;
  if (!offsets_ok(pen->hist_off, b)) return ST_BAD_OFFSETS;
  for (int32_t h = pen->hist_off[b]; h < pen->hist_off[b + 1]; ++h)
    if (pen->hist_cols[h] < 0 || pen->hist_cols[h] >= V) return ST_ID_RANGE;
  return 0;
}

void tto_align(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
               const int32_t* target_off, const int32_t* target_ids,
               const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
               const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
               int32_t w, int32_t* path, int32_t* path_len, int32_t* cost,
               int32_t* map, int32_t* status) {
  for (int32_t b = 0; b < B; ++b) {
    path_len[b] = 0;
    cost[b] = -1;
    if (!offsets_ok(draft_off, b) || !offsets_ok(target_off, b)) {
      status[b] = ST_BAD_OFFSETS;
      continue;
    }
    int32_t d0 = draft_off[b], k = draft_off[b + 1] - d0;
    int32_t t0 = target_off[b], m = target_off[b + 1] - t0;
    int32_t st = 0;
    for (int32_t j = 0; j < m; ++j) map[t0 + j] = -1;
    if (k == 0 || m == 0) st |= ST_EMPTY;
    if (k > MAX_K || m > MAX_M) st |= ST_TOO_LONG;
    /* length checks first; only then every token is looked at, OR-ing flags */
    int32_t skip_tokens = st != 0;
    for (int32_t i = 0; i < k && !skip_tokens; ++i) {
      int32_t id = draft_ids[d0 + i];
      if (id < 0 || id >= Vd) st |= ST_ID_RANGE;
      else if (vd_off[id + 1] - vd_off[id] > MAX_TOKEN_BYTES) st |= ST_TOO_LONG;
    }
    for (int32_t j = 0; j < m && !skip_tokens; ++j) {
      int32_t id = target_ids[t0 + j];
      if (id < 0 || id >= Vt) st |= ST_ID_RANGE;
      else if (vt_off[id + 1] - vt_off[id] > MAX_TOKEN_BYTES) st |= ST_TOO_LONG;
    }
    status[b] = st;
    if (st) continue;
    /* local cost d(x_i, y_j) for every cell (the band only reads some) */
    int32_t* d = (int32_t*)malloc(sizeof(int32_t) * (size_t)k * (size_t)m);
    for (int32_t i = 0; i < k; ++i) {
      int32_t a = draft_ids[d0 + i];
      for (int32_t j = 0; j < m; ++j) {
        int32_t c = target_ids[t0 + j];
        d[(int64_t)i * m + j] =
            tto_lev(vd_bytes + vd_off[a], (int32_t)(vd_off[a + 1] - vd_off[a]),
                    vt_bytes + vt_off[c], (int32_t)(vt_off[c + 1] - vt_off[c]));
      }
    }
    int32_t* pb = path + 2 * ((int64_t)d0 + t0);
    int32_t L = 0;
    int64_t cs = tto_dtw(k, m, d, w, pb, &L);
    free(d);
    path_len[b] = L;
    cost[b] = (int32_t)cs;
    /* map[j] = largest draft index aligned to target index j */
    for (int32_t x = 0; x < L; ++x) {
      int32_t i = pb[2 * x], j = pb[2 * x + 1];
      if (i > map[t0 + j]) map[t0 + j] = i;
    }
  }
}

/* ---------------------------------------------------------------- transfer */

/* The transfer with the draft rows' filters; drow_bnd (may be NULL) gets bit 4
 * for each draft row whose top-p cut is ambiguous (the request-wide bit of
 * `boundary` is the OR of its rows'). */
static void transfer_impl(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                          const int32_t* target_off, const int32_t* map,
                          const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                          const float* draft_probs, double T_d, int32_t top_k, double top_p,
                          double* q_hat, int32_t* status, int32_t* boundary,
                          int32_t* drow_bnd, const tto_penalty* pen) {
  const int filtered = top_k > 0 || (top_p > 0.0 && top_p < 1.0);
  double* qf = filtered ? (double*)malloc(sizeof(double) * (size_t)(V > 0 ? V : 1)) : NULL;
  const int penal = pen && pen->theta != 1.0f && !draft_probs;
  float* pbuf = penal ? (float*)malloc(sizeof(float) * (size_t)(V > 0 ? V : 1)) : NULL;
  uint8_t* mark = penal ? (uint8_t*)malloc((size_t)(V > 0 ? V : 1)) : NULL;
  for (int32_t b = 0; b < B; ++b) {
    if (boundary) boundary[b] = 0;
    if (!offsets_ok(draft_off, b) || !offsets_ok(target_off, b)) {
      status[b] = ST_BAD_OFFSETS;
      continue;
    }
    int32_t d0 = draft_off[b], k = draft_off[b + 1] - d0;
    int32_t t0 = target_off[b], m = target_off[b + 1] - t0;
    int32_t st = 0;
    if (k == 0 || m == 0) st |= ST_EMPTY;
    int32_t skip_tokens = st != 0;
    for (int32_t j = 0; j < m && !skip_tokens; ++j)
      if (map[t0 + j] < 0 || map[t0 + j] >= k) st |= ST_ID_RANGE;
    for (int32_t i = 0; i < k && !skip_tokens && !draft_probs; ++i)
      if (draft_cols[d0 + i] < 0 || draft_cols[d0 + i] >= V) st |= ST_ID_RANGE;
    if (!st && penal) st |= history_status(pen, b, V);
    status[b] = st;
    for (int32_t j = 0; j < m; ++j) q_hat[t0 + j] = 0.0;
    if (st) continue;
    int64_t have = -1; /* the draft row whose filtered distribution qf holds */
    for (int32_t j = 0; j < m; ++j) {
      int64_t r = (int64_t)d0 + map[t0 + j];
      if (draft_probs) {
        q_hat[t0 + j] = (double)draft_probs[r];
        continue;
      }
      /* draft row map[j] scores d_{map[j]+1}: the draft tokens before it are penalized */
      int32_t rdt = dtype;
      const void* row = penalized_row(row_ptr(draft_logits, dtype, row_stride, r), dtype, V,
                                      penal ? pen : NULL, b, draft_cols + d0, map[t0 + j], pbuf,
                                      mark, &rdt);
      if (filtered) {
        if (r != have) {
          int32_t rb = 0;
          tto_filtered_probs(row, rdt, V, T_d, top_k, top_p, qf, &rb);
          if (boundary) boundary[b] |= rb;
          if (drow_bnd) drow_bnd[r] |= rb;
          have = r;
        }
        q_hat[t0 + j] = qf[draft_cols[r]];
      } else {
        double lse = tto_logsumexp(row, rdt, V, T_d);
        q_hat[t0 + j] = exp(load_logit(row, rdt, draft_cols[r]) / T_d - lse);
      }
    }
  }
  free(qf);
  free(pbuf);
  free(mark);
}

void tto_transfer2(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                   const int32_t* target_off, const int32_t* map,
                   const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                   const float* draft_probs, double T_d, int32_t top_k, double top_p,
                   double* q_hat, int32_t* status, int32_t* boundary) {
  transfer_impl(B, draft_off, draft_cols, target_off, map, draft_logits, dtype, row_stride, V,
                draft_probs, T_d, top_k, top_p, q_hat, status, boundary, NULL, NULL);
}

void tto_transfer3(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                   const int32_t* target_off, const int32_t* map,
                   const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                   const float* draft_probs, double T_d, int32_t top_k, double top_p,
                   double* q_hat, int32_t* status, int32_t* boundary, int32_t* drow_bnd) {
  transfer_impl(B, draft_off, draft_cols, target_off, map, draft_logits, dtype, row_stride, V,
                draft_probs, T_d, top_k, top_p, q_hat, status, boundary, drow_bnd, NULL);
}

void tto_transfer_pen(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                      const int32_t* target_off, const int32_t* map,
                      const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                      const float* draft_probs, double T_d, int32_t top_k, double top_p,
                      const tto_penalty* pen, double* q_hat, int32_t* status, int32_t* boundary,
                      int32_t* drow_bnd) {
  transfer_impl(B, draft_off, draft_cols, target_off, map, draft_logits, dtype, row_stride, V,
                draft_probs, T_d, top_k, top_p, q_hat, status, boundary, drow_bnd, pen);
}

void tto_transfer(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                  const int32_t* target_off, const int32_t* map,
                  const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                  const float* draft_probs, double T_d, double* q_hat, int32_t* status) {
  tto_transfer2(B, draft_off, draft_cols, target_off, map, draft_logits, dtype, row_stride, V,
                draft_probs, T_d, 0, 1.0, q_hat, status, NULL);
}

/* ------------------------------------------------------------------ verify */

/* The verification; besides the request-wide boundary bits it can report
 * where each one lies (all three may be NULL): row_bnd[r] for every target row
 * r (indexed as lse) gets bit 1 when the accept decision of the position that
 * row scores lay within 1e-6 of its threshold, bit 4 when the row's top-p cut
 * is ambiguous, bit 8 (full-q) when the kept set of the draft row that the
 * residual of this row subtracts is ambiguous; tok_lo[b] / tok_hi[b] are the
 * first and last column of the drawn row whose running mass lies within
 * 1e-6 Z of u' Z (-1 when none). None of these changes any result. */
static void verify_impl(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                        const double* q_hat, const void* target_logits, int32_t dtype_t,
                        int64_t stride_t, int32_t V_t, double T_t,
                        const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                        int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                        int32_t full_q, uint64_t seed, uint64_t request_base,
                        int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                        int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                        int32_t* status, int32_t* boundary, int32_t* row_bnd,
                        int32_t* tok_lo, int32_t* tok_hi, const tto_penalty* pen_t) {
  const int filt_t = top_k_t > 0 || (top_p_t > 0.0 && top_p_t < 1.0);
  const int filt_d = top_k_d > 0 || (top_p_d > 0.0 && top_p_d < 1.0);
  const int penal = pen_t && pen_t->theta != 1.0f;
  float* pbuf = penal ? (float*)malloc(sizeof(float) * (size_t)V_t) : NULL;
  uint8_t* mark = penal ? (uint8_t*)malloc((size_t)V_t) : NULL;
  double* pf = filt_t ? (double*)malloc(sizeof(double) * (size_t)V_t) : NULL;
  double* p = (double*)malloc(sizeof(double) * (size_t)V_t);
  double* q = full_q ? (double*)malloc(sizeof(double) * (size_t)V_d) : NULL;
  double* r = (double*)malloc(sizeof(double) * (size_t)V_t);
  for (int32_t b = 0; b < B; ++b) {
    accepted[b] = 0;
    next_token[b] = -1;
    boundary[b] = 0;
    if (tok_lo) tok_lo[b] = -1;
    if (tok_hi) tok_hi[b] = -1;
    if (!offsets_ok(target_off, b)) {
      status[b] = ST_BAD_OFFSETS;
      continue;
    }
    int32_t t0 = target_off[b], m = target_off[b + 1] - t0;
    int64_t row0 = (int64_t)t0 + b; /* request b owns target rows row0 .. row0+m */
    int32_t st = 0;
    if (m == 0) st |= ST_EMPTY;
    if (m > MAX_M) st |= ST_TOO_LONG;
    int32_t skip_tokens = st != 0;
    for (int32_t j = 0; j < m && !skip_tokens; ++j)
      if (target_cols[t0 + j] < 0 || target_cols[t0 + j] >= V_t) st |= ST_ID_RANGE;
    if (full_q && !skip_tokens) {
      if (!offsets_ok(draft_off, b)) {
        st |= ST_BAD_OFFSETS;
      } else {
        int32_t k = draft_off[b + 1] - draft_off[b];
        if (k == 0) st |= ST_EMPTY;
        for (int32_t j = 0; j < m && k > 0; ++j)
          if (map[t0 + j] < 0 || map[t0 + j] >= k) st |= ST_ID_RANGE;
      }
    }
    if (!st && penal) st |= history_status(pen_t, b, V_t);
    status[b] = st;
    if (st) continue;

    /* p_hat_j = p_j(t_j) for every target position; lse of all m+1 rows
       (with filters: of the kept set); row j scores t_{j+1}, so with a
       penalty the proxy tokens t_1..t_j join the request's history */
    for (int32_t j = 0; j <= m; ++j) {
      int32_t rdt = dtype_t;
      const void* row = penalized_row(row_ptr(target_logits, dtype_t, stride_t, row0 + j),
                                      dtype_t, V_t, pen_t, b, target_cols + t0, j, pbuf, mark,
                                      &rdt);
      if (filt_t) {
        int32_t rb = 0;
        double l = tto_filtered_probs(row, rdt, V_t, T_t, top_k_t, top_p_t, pf, &rb);
        boundary[b] |= rb;
        if (row_bnd) row_bnd[row0 + j] |= rb;
        if (lse) lse[row0 + j] = l;
        if (j < m) p_hat[t0 + j] = pf[target_cols[t0 + j]];
      } else {
        double l = tto_logsumexp(row, rdt, V_t, T_t);
        if (lse) lse[row0 + j] = l;
        if (j < m) p_hat[t0 + j] = exp(load_logit(row, rdt, target_cols[t0 + j]) / T_t - l);
      }
    }

    /* sequential accept, stop at the first rejection */
    int32_t a = 0;
    for (int32_t j = 0; j < m; ++j) {
      double u = tto_uniform(seed, (uint64_t)j, 0, request_base + (uint64_t)b);
      double ph = p_hat[t0 + j], qh = q_hat[t0 + j];
      double ratio = qh > 0.0 ? ph / qh : (ph > 0.0 ? INFINITY : 0.0);
      double acc = ratio < 1.0 ? ratio : 1.0;
      if (fabs(u - acc) < BOUNDARY_EPS) {
        boundary[b] |= 1;
        if (row_bnd) row_bnd[row0 + j] |= 1;
      }
      if (u < acc) ++a;
      else break;
    }
    accepted[b] = a;

    /* the residual (or bonus) row a */
    int32_t pdt = dtype_t;
    const void* prow = penalized_row(row_ptr(target_logits, dtype_t, stride_t, row0 + a),
                                     dtype_t, V_t, pen_t, b, target_cols + t0, a, pbuf, mark,
                                     &pdt);
    if (filt_t) tto_filtered_probs(prow, pdt, V_t, T_t, top_k_t, top_p_t, p, &boundary[b]);
    else tto_softmax(prow, pdt, V_t, T_t, p);
    if (a < m) {
      if (full_q) {
        const void* qrow = row_ptr(draft_logits, dtype_d, stride_d,
                                   (int64_t)draft_off[b] + map[t0 + a]);
        if (filt_d) {
          int32_t rb = 0;
          tto_filtered_probs(qrow, dtype_d, V_d, T_d, top_k_d, top_p_d, q, &rb);
          boundary[b] |= rb;
          if (row_bnd && rb) row_bnd[row0 + a] |= 8;
        } else {
          tto_softmax(qrow, dtype_d, V_d, T_d, q);
        }
        for (int32_t x = 0; x < V_t; ++x) r[x] = p[x] > q[x] ? p[x] - q[x] : 0.0;
      } else {
        int32_t t = target_cols[t0 + a];
        for (int32_t x = 0; x < V_t; ++x) r[x] = p[x];
        double rt = p[t] - q_hat[t0 + a];
        r[t] = rt > 0.0 ? rt : 0.0;
      }
    } else {
      for (int32_t x = 0; x < V_t; ++x) r[x] = p[x];
    }
    double Z = 0.0;
    for (int32_t x = 0; x < V_t; ++x) Z += r[x];
    if (!(Z > 0.0)) { /* degenerate residual: fall back to the row itself */
      for (int32_t x = 0; x < V_t; ++x) r[x] = p[x];
      Z = 0.0;
      for (int32_t x = 0; x < V_t; ++x) Z += r[x];
    }
    double u2 = tto_uniform(seed, (uint64_t)a, 1, request_base + (uint64_t)b);
    double theta = u2 * Z, cum = 0.0;
    int32_t pick = -1, last_pos = -1;
    for (int32_t x = 0; x < V_t; ++x) {
      cum += r[x];
      if (r[x] > 0.0) last_pos = x;
      if (fabs(theta - cum) < BOUNDARY_EPS * Z) {
        boundary[b] |= 2;
        if (tok_lo && tok_lo[b] < 0) tok_lo[b] = x;
        if (tok_hi) tok_hi[b] = x;
      }
      if (pick < 0 && cum > theta) pick = x;
    }
    next_token[b] = pick >= 0 ? pick : last_pos;
  }
  free(p);
  free(q);
  free(r);
  free(pf);
  free(pbuf);
  free(mark);
}

void tto_verify2(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                 const double* q_hat, const void* target_logits, int32_t dtype_t,
                 int64_t stride_t, int32_t V_t, double T_t,
                 const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                 int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                 int32_t full_q, uint64_t seed, uint64_t request_base,
                 int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                 int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                 int32_t* status, int32_t* boundary) {
  verify_impl(B, target_off, target_cols, q_hat, target_logits, dtype_t, stride_t, V_t, T_t,
              draft_off, map, draft_logits, dtype_d, stride_d, V_d, T_d, full_q, seed,
              request_base, top_k_t, top_p_t, top_k_d, top_p_d, accepted, next_token, p_hat,
              lse, status, boundary, NULL, NULL, NULL, NULL);
}

void tto_verify3(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                 const double* q_hat, const void* target_logits, int32_t dtype_t,
                 int64_t stride_t, int32_t V_t, double T_t,
                 const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                 int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                 int32_t full_q, uint64_t seed, uint64_t request_base,
                 int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                 int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                 int32_t* status, int32_t* boundary, int32_t* row_bnd, int32_t* tok_lo,
                 int32_t* tok_hi) {
  verify_impl(B, target_off, target_cols, q_hat, target_logits, dtype_t, stride_t, V_t, T_t,
              draft_off, map, draft_logits, dtype_d, stride_d, V_d, T_d, full_q, seed,
              request_base, top_k_t, top_p_t, top_k_d, top_p_d, accepted, next_token, p_hat,
              lse, status, boundary, row_bnd, tok_lo, tok_hi, NULL);
}

void tto_verify_pen(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                    const double* q_hat, const void* target_logits, int32_t dtype_t,
                    int64_t stride_t, int32_t V_t, double T_t,
                    const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                    int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                    int32_t full_q, uint64_t seed, uint64_t request_base,
                    int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                    const tto_penalty* pen_t, int32_t* accepted, int32_t* next_token,
                    double* p_hat, double* lse, int32_t* status, int32_t* boundary,
                    int32_t* row_bnd, int32_t* tok_lo, int32_t* tok_hi) {
  verify_impl(B, target_off, target_cols, q_hat, target_logits, dtype_t, stride_t, V_t, T_t,
              draft_off, map, draft_logits, dtype_d, stride_d, V_d, T_d, full_q, seed,
              request_base, top_k_t, top_p_t, top_k_d, top_p_d, accepted, next_token, p_hat,
              lse, status, boundary, row_bnd, tok_lo, tok_hi, pen_t);
}

void tto_verify(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                const double* q_hat, const void* target_logits, int32_t dtype_t,
                int64_t stride_t, int32_t V_t, double T_t,
                const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                int32_t full_q, uint64_t seed, uint64_t request_base,
                int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                int32_t* status, int32_t* boundary) {
  tto_verify2(B, target_off, target_cols, q_hat, target_logits, dtype_t, stride_t, V_t, T_t,
              draft_off, map, draft_logits, dtype_d, stride_d, V_d, T_d, full_q, seed,
              request_base, 0, 1.0, 0, 1.0, accepted, next_token, p_hat, lse, status, boundary);
}

/* ------------------------------------------------------------ re-encoding */

/* The target vocabulary sorted by (byte string, id), so that a string's
 * smallest id is the first of its run. The sort's comparator reads the table
 * through these file-level pointers (the oracle is single-threaded). */
static const uint8_t* g_sort_bytes;
static const int64_t* g_sort_off;

static int cmp_bytes(const uint8_t* a, int64_t na, const uint8_t* b, int64_t nb) {
  int64_t n = na < nb ? na : nb;
  int c = n > 0 ? memcmp(a, b, (size_t)n) : 0;
  if (c != 0) return c;
  return na < nb ? -1 : (na > nb ? 1 : 0);
}

static int cmp_token_ids(const void* x, const void* y) {
  int32_t a = *(const int32_t*)x, b = *(const int32_t*)y;
  int c = cmp_bytes(g_sort_bytes + g_sort_off[a], g_sort_off[a + 1] - g_sort_off[a],
                    g_sort_bytes + g_sort_off[b], g_sort_off[b + 1] - g_sort_off[b]);
  if (c != 0) return c;
  return a < b ? -1 : (a > b ? 1 : 0);
}

/* Smallest id of vt spelling s[0..n), or -1 (binary search over the sorted ids). */
static int32_t find_token(const int32_t* sorted, int32_t Vt, const uint8_t* vt_bytes,
                          const int64_t* vt_off, const uint8_t* s, int64_t n) {
  int32_t lo = 0, hi = Vt;  /* first position whose string is >= s */
  while (lo < hi) {
    int32_t mid = lo + (hi - lo) / 2;
    int32_t v = sorted[mid];
    if (cmp_bytes(vt_bytes + vt_off[v], vt_off[v + 1] - vt_off[v], s, n) < 0) lo = mid + 1;
    else hi = mid;
  }
  if (lo < Vt) {
    int32_t v = sorted[lo];
    if (cmp_bytes(vt_bytes + vt_off[v], vt_off[v + 1] - vt_off[v], s, n) == 0) return v;
  }
  return -1;
}

void tto_encode(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
                const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
                const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
                int32_t max_m, int32_t max_bytes, int32_t capacity,
                int32_t* target_off, int32_t* target_ids, int32_t* status) {
  int32_t* sorted = (int32_t*)malloc(sizeof(int32_t) * (size_t)(Vt > 0 ? Vt : 1));
  int64_t longest = 0;
  for (int32_t v = 0; v < Vt; ++v) {
    sorted[v] = v;
    if (vt_off[v + 1] - vt_off[v] > longest) longest = vt_off[v + 1] - vt_off[v];
  }
  g_sort_bytes = vt_bytes;
  g_sort_off = vt_off;
  qsort(sorted, (size_t)Vt, sizeof(int32_t), cmp_token_ids);

  uint8_t* text = (uint8_t*)malloc((size_t)(max_bytes > 0 ? max_bytes : 1));
  int32_t* toks = (int32_t*)malloc(sizeof(int32_t) * (size_t)(max_m > 0 ? max_m : 1));
  int64_t end_all = 0; /* tokens of every earlier request, written or not */
  target_off[0] = 0;
  for (int32_t b = 0; b < B; ++b) {
    int32_t st = 0, m = 0;
    if (!offsets_ok(draft_off, b)) {
      st = ST_BAD_OFFSETS;
    } else {
      int32_t d0 = draft_off[b], k = draft_off[b + 1] - d0;
      int64_t n = 0;
      if (k == 0) st |= ST_EMPTY;
      for (int32_t i = 0; i < k; ++i) {
        int32_t id = draft_ids[d0 + i];
        if (id < 0 || id >= Vd) { st |= ST_ID_RANGE; continue; }
        n += vd_off[id + 1] - vd_off[id];
      }
      if (st == 0 && n > max_bytes) st |= ST_TOO_LONG;
      if (st == 0) {
        /* decode_d: concatenate the draft tokens' bytes */
        int64_t at = 0;
        for (int32_t i = 0; i < k; ++i) {
          int32_t id = draft_ids[d0 + i];
          int64_t len = vd_off[id + 1] - vd_off[id];
          if (len > 0) memcpy(text + at, vd_bytes + vd_off[id], (size_t)len);
          at += len;
        }
        /* encode_t: greedy longest match */
        int64_t p = 0;
        while (p < n && st == 0) {
          int64_t L = n - p < longest ? n - p : longest;
          int32_t v = -1;
          for (; L >= 1; --L) {
            v = find_token(sorted, Vt, vt_bytes, vt_off, text + p, L);
            if (v >= 0) break;
          }
          if (v < 0) { st |= ST_NO_MATCH; break; }
          if (m >= max_m) { st |= ST_TOO_LONG; break; }
          toks[m++] = v;
          p += L;
        }
      }
    }
    if (st != 0) m = 0;
    end_all += m;
    if (st == 0 && end_all > capacity) { st |= ST_TOO_LONG; m = 0; }
    for (int32_t j = 0; j < m; ++j) target_ids[target_off[b] + j] = toks[j];
    target_off[b + 1] = target_off[b] + m;
    status[b] = st;
  }
  free(text);
  free(toks);
  free(sorted);
}

void tto_consistency(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
                     const int32_t* target_off, const int32_t* target_ids,
                     const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
                     const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
                     int32_t max_k, int32_t max_m, int32_t* status) {
  for (int32_t b = 0; b < B; ++b) {
    if (!offsets_ok(draft_off, b) || !offsets_ok(target_off, b)) {
      status[b] = ST_BAD_OFFSETS;
      continue;
    }
    int32_t d0 = draft_off[b], k = draft_off[b + 1] - d0;
    int32_t t0 = target_off[b], m = target_off[b + 1] - t0;
    int32_t st = 0;
    if (k > max_k || m > max_m) st |= ST_TOO_LONG;
    for (int32_t i = 0; i < k; ++i)
      if (draft_ids[d0 + i] < 0 || draft_ids[d0 + i] >= Vd) st |= ST_ID_RANGE;
    for (int32_t j = 0; j < m; ++j)
      if (target_ids[t0 + j] < 0 || target_ids[t0 + j] >= Vt) st |= ST_ID_RANGE;
    if (st == 0) {
      /* walk both byte streams side by side */
      int32_t i = 0, j = 0;
      int64_t pi = 0, pj = 0; /* position inside token i / token j */
      for (;;) {
        while (i < k && pi == vd_off[draft_ids[d0 + i] + 1] - vd_off[draft_ids[d0 + i]]) {
          ++i;
          pi = 0;
        }
        while (j < m && pj == vt_off[target_ids[t0 + j] + 1] - vt_off[target_ids[t0 + j]]) {
          ++j;
          pj = 0;
        }
        if (i == k || j == m) {
          if (i != k || j != m) st |= ST_INCONSISTENT; /* one string is longer */
          break;
        }
        if (vd_bytes[vd_off[draft_ids[d0 + i]] + pi] != vt_bytes[vt_off[target_ids[t0 + j]] + pj]) {
          st |= ST_INCONSISTENT;
          break;
        }
        ++pi;
        ++pj;
      }
    }
    status[b] = st;
  }
}

void tto_dpos_hist(int32_t B, const int32_t* draft_off, const int32_t* target_off,
                   const int32_t* path, const int32_t* path_len, const int32_t* map,
                   int32_t mode, int32_t n_bins, int64_t* hist) {
  for (int32_t b = 0; b < B; ++b) {
    if (path_len[b] <= 0) continue;
    if (mode == 0) {
      const int32_t* pp = path + 2 * ((int64_t)draft_off[b] + target_off[b]);
      for (int32_t x = 0; x < path_len[b]; ++x) {
        int32_t d = abs(pp[2 * x] - pp[2 * x + 1]);
        hist[d < n_bins - 1 ? d : n_bins - 1] += 1;
      }
    } else {
      for (int32_t j = 0; j < target_off[b + 1] - target_off[b]; ++j) {
        int32_t d = abs(map[target_off[b] + j] - j);
        hist[d < n_bins - 1 ? d : n_bins - 1] += 1;
      }
    }
  }
}
