/*
 * tto.h -- CPU oracle of the TokenTiming verification path (arXiv 2510.15545).
 *
 * TEST INFRASTRUCTURE. This library is the slow, plain reference that the CUDA
 * path is compared against. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline / reference legs load it; the product path never
 * does. It shares no code, header or constant with the CUDA library.
 *
 * Arithmetic is fp64 throughout; every routine is the textbook form of the
 * passage it cites. Indices are 0-based in all arrays.
 *
 * Per-request status bits (the same values the CUDA library documents):
 *   1 id out of range, 2 too long, 4 empty request, 8 bad CSR offsets.
 * Boundary bits (oracle only): 1 = some accept draw u_j lay within 1e-6 of
 * min(1, p/q); 2 = the residual draw u' lay within 1e-6 of a CDF breakpoint.
 */
#ifndef TTO_H
#define TTO_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* App. H: Levenshtein distance between byte strings, unit costs. */
int32_t tto_lev(const uint8_t* s, int32_t ns, const uint8_t* t, int32_t nt);

/* Alg. 1 on a given k x m local cost matrix d (row-major, d[i*m+j] =
 * d(x_{i+1}, y_{j+1})). w < 0: no band. Writes the optimal path as 0-based
 * (i, j) pairs in forward order (capacity k+m pairs) and returns C* (or -1). */
int64_t tto_dtw(int32_t k, int32_t m, const int32_t* d, int32_t w,
                int32_t* path, int32_t* path_len);

/* Philox4x64-10 (Salmon et al., SC'11) of one counter block. */
void tto_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2], uint64_t out[4]);

/* Uniform in [0,1): top 24 bits of the first Philox word times 2^-24, for
 * counter (pos, stream, request, 0) and key (seed, 0). */
double tto_uniform(uint64_t seed, uint64_t pos, uint64_t stream, uint64_t request);

/* Two-pass fp64 softmax of row/T (row: fp32 or bf16 values, dtype 0 / 1). */
void tto_softmax(const void* row, int32_t dtype, int64_t V, double T, double* p_out);
double tto_logsumexp(const void* row, int32_t dtype, int64_t V, double T);

/* Batched DTW alignment (§4.1, Alg. 1, App. H). Outputs are per request:
 * path pairs at pair offset draft_off[b] + target_off[b], path_len[b],
 * cost[b] = C*, map[j] = max{i : (i,j) on the path} for the request's target
 * positions, status[b]. */
void tto_align(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
               const int32_t* target_off, const int32_t* target_ids,
               const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
               const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
               int32_t w, int32_t* path, int32_t* path_len, int32_t* cost,
               int32_t* map, int32_t* status);

/* MapProbabilities (Alg. 2, App. A.2): q_hat[j] = probability of the mapped
 * draft token d_{map[j]} under its own draft row at temperature T_d, or
 * draft_probs[row] when draft_probs is not NULL. */
void tto_transfer(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                  const int32_t* target_off, const int32_t* map,
                  const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                  const float* draft_probs, double T_d, double* q_hat, int32_t* status);

/* Verification (Alg. 2 accept loop, Alg. 4 residual): accept target token j
 * while u_j < min(1, p_j / q_hat_j); then sample the next token from the
 * normalised residual of row a (or from the bonus row when all m were
 * accepted). full_q != 0: homogeneous vocabulary, residual max(0, p - q) with
 * q the full draft row map[a]. */
void tto_verify(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                const double* q_hat, const void* target_logits, int32_t dtype_t,
                int64_t stride_t, int32_t V_t, double T_t,
                const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                int32_t full_q, uint64_t seed, uint64_t request_base,
                int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                int32_t* status, int32_t* boundary);

/* ------------------------------------------------------- sampling filters */

/* Temperature, then top-k (keep the k largest logits, smaller column first
 * among equal ones; k <= 0 or k >= V: none), then top-p (keep tokens in
 * decreasing probability while the mass before a token is below top_p; top_p
 * <= 0 or >= 1: none), as in the paper's generation hyperparameters. Writes the
 * filtered distribution over all V columns and returns the log of the kept
 * set's normaliser. *boundary (may be NULL) gets bit 4 when the mass before
 * some token lies within 1e-6 of top_p. */
double tto_filtered_probs(const void* row, int32_t dtype, int64_t V, double T, int32_t top_k,
                          double top_p, double* p, int32_t* boundary);

/* tto_transfer with the draft rows' filters (boundary: bit 4 as above, may be NULL). */
void tto_transfer2(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                   const int32_t* target_off, const int32_t* map,
                   const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                   const float* draft_probs, double T_d, int32_t top_k, double top_p,
                   double* q_hat, int32_t* status, int32_t* boundary);

/* tto_verify with filters on the target rows (p) and, in full-q mode, on the
 * draft rows (q); lse is then the log-normaliser of each target row's kept set. */
void tto_verify2(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                 const double* q_hat, const void* target_logits, int32_t dtype_t,
                 int64_t stride_t, int32_t V_t, double T_t,
                 const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                 int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                 int32_t full_q, uint64_t seed, uint64_t request_base,
                 int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                 int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                 int32_t* status, int32_t* boundary);

/* tto_transfer2 that also says which draft rows have an ambiguous top-p cut:
 * drow_bnd[r] (n_draft entries, OR-ed into: the caller clears it) gets bit 4
 * for each such row r. Results are those of tto_transfer2. */
void tto_transfer3(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                   const int32_t* target_off, const int32_t* map,
                   const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                   const float* draft_probs, double T_d, int32_t top_k, double top_p,
                   double* q_hat, int32_t* status, int32_t* boundary, int32_t* drow_bnd);

/* tto_verify2 that also says where each boundary case lies, so that a
 * comparison can excuse a difference only at the decision it concerns.
 * row_bnd (n_target + B entries, indexed as lse, OR-ed into: the caller clears
 * it): bit 1 = the accept decision of the position this row scores lay within
 * 1e-6 of min(1, p/q); bit 4 = this row's top-p cut is ambiguous; bit 8 =
 * full-q, the kept set of the draft row the residual of this row subtracts is
 * ambiguous. tok_lo[b] / tok_hi[b]: first and last column of the drawn row
 * whose running mass lies within 1e-6 Z of u' Z, -1 when none. Results are
 * those of tto_verify2. */
void tto_verify3(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                 const double* q_hat, const void* target_logits, int32_t dtype_t,
                 int64_t stride_t, int32_t V_t, double T_t,
                 const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                 int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                 int32_t full_q, uint64_t seed, uint64_t request_base,
                 int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                 int32_t* accepted, int32_t* next_token, double* p_hat, double* lse,
                 int32_t* status, int32_t* boundary, int32_t* row_bnd, int32_t* tok_lo,
                 int32_t* tok_hi);

/* ------------------------------------------------------ repetition penalty */

/* The repetition penalty of the generation hyperparameters (App. F): a request's
 * history of logits columns (hist_cols[hist_off[b] .. hist_off[b+1]), CSR; NULL
 * hist_off = empty histories) and the penalty theta (1 = off). A row's
 * penalized set is the history plus the sequence tokens before the row's
 * position (target row j: t_1..t_j; draft row i: d_1..d_i, 0-based rows);
 * each of its columns has z replaced by z * theta when z < 0, else by
 * z / theta, in fp32, before temperature and the filters. A history column
 * out of range gives status 1, a bad history range status 8. */
typedef struct {
  const int32_t* hist_off;
  const int32_t* hist_cols;
  float theta;
} tto_penalty;

/* tto_transfer3 with a penalty on the draft rows (NULL: none; ignored with
 * given draft probabilities). */
void tto_transfer_pen(int32_t B, const int32_t* draft_off, const int32_t* draft_cols,
                      const int32_t* target_off, const int32_t* map,
                      const void* draft_logits, int32_t dtype, int64_t row_stride, int32_t V,
                      const float* draft_probs, double T_d, int32_t top_k, double top_p,
                      const tto_penalty* pen, double* q_hat, int32_t* status, int32_t* boundary,
                      int32_t* drow_bnd);

/* tto_verify3 with a penalty on the target rows (NULL: none). */
void tto_verify_pen(int32_t B, const int32_t* target_off, const int32_t* target_cols,
                    const double* q_hat, const void* target_logits, int32_t dtype_t,
                    int64_t stride_t, int32_t V_t, double T_t,
                    const int32_t* draft_off, const int32_t* map, const void* draft_logits,
                    int32_t dtype_d, int64_t stride_d, int32_t V_d, double T_d,
                    int32_t full_q, uint64_t seed, uint64_t request_base,
                    int32_t top_k_t, double top_p_t, int32_t top_k_d, double top_p_d,
                    const tto_penalty* pen_t, int32_t* accepted, int32_t* next_token,
                    double* p_hat, double* lse, int32_t* status, int32_t* boundary,
                    int32_t* row_bnd, int32_t* tok_lo, int32_t* tok_hi);

/* ------------------------------------------------------------ re-encoding */

/* Re-encoding (§4.2; App. A.1, Lemma 1): T_b = encode_t(decode_d(D_b)).
 * decode_d concatenates the byte strings of the draft tokens; encode_t is
 * greedy longest match over vt: at each position the longest token of vt that
 * spells the next bytes (the smallest id among tokens with equal strings;
 * empty tokens never match). Per request: status 8 bad draft offsets, 1 a
 * draft id out of range, 4 no draft token, 2 decoded string longer than
 * max_bytes or more than max_m target tokens, 128 some position that no token
 * of vt spells. A request that fails writes no tokens. Requests are laid out in
 * order in target_ids; a request whose tokens would end past `capacity`
 * (counting every earlier request's tokens, written or not) is not written and
 * gets status 2. target_off[b+1] = target_off[b] + (tokens written for b). */
void tto_encode(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
                const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
                const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
                int32_t max_m, int32_t max_bytes, int32_t capacity,
                int32_t* target_off, int32_t* target_ids, int32_t* status);

/* Lemma 1 (App. A.1) as a check: decode_t(T_b) == decode_d(D_b) byte for byte.
 * Status bits: 8 bad offsets, 1 id out of range, 2 k > max_k or m > max_m,
 * 256 the two byte strings differ. */
void tto_consistency(int32_t B, const int32_t* draft_off, const int32_t* draft_ids,
                     const int32_t* target_off, const int32_t* target_ids,
                     const uint8_t* vd_bytes, const int64_t* vd_off, int32_t Vd,
                     const uint8_t* vt_bytes, const int64_t* vt_off, int32_t Vt,
                     int32_t max_k, int32_t max_m, int32_t* status);

/* Delta-pos (§4.1, App. K): the position deviation |i - j| of matched tokens,
 * counted into hist[min(|i - j|, n_bins - 1)] (hist is added to, not cleared).
 * mode 0: every (i, j) on each request's DTW path; mode 1: every target
 * position j with its mapped draft index map[j]. Requests with path_len[b] == 0
 * (failed alignments) add nothing. */
void tto_dpos_hist(int32_t B, const int32_t* draft_off, const int32_t* target_off,
                   const int32_t* path, const int32_t* path_len, const int32_t* map,
                   int32_t mode, int32_t n_bins, int64_t* hist);

#ifdef __cplusplus
}
#endif
#endif
