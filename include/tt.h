/*
 * tt.h -- C ABI of the TokenTiming verification hot path on one NVIDIA GB300
 * (sm_103a). TokenTiming: arXiv 2510.15545 ("TokenTiming: A Dynamic Alignment
 * Method for Universal Speculative Decoding Model Pairs").
 *
 * One verification step of a batch of B independent requests:
 *   (a) align   -- Dynamic Token Warping (§4.1, Alg. 1) between each request's
 *                  draft tokens D = (d_1..d_k) and its proxy target tokens
 *                  T = (t_1..t_m) = encode_t(decode_d(D)) (§4.2, App. A.1),
 *                  with the Levenshtein distance over the tokens' UTF-8 bytes as
 *                  the local cost (App. H) and a Sakoe-Chiba band (§4.1);
 *   (b) transfer -- MapProbabilities (Alg. 2, App. A.2): target position j
 *                  takes the draft probability of the last draft token aligned
 *                  to it (terminal rule / copy rule), one-hot (Limitations);
 *   (c) verify  -- speculative sampling (§4.2 verification, Alg. 4): accept t_j
 *                  while u_j < min(1, p(t_j)/q(t_j)), stop at the first
 *                  rejection, then draw the next token from the normalised
 *                  residual max(0, p - q) over the whole target vocabulary (or
 *                  from the bonus row m+1 when all m were accepted).
 * Here p is the target distribution and q the draft one (Alg. 4's naming).
 *
 * Conventions shared by every entry point:
 *  - Every pointer is a DEVICE pointer owned by the caller, unless stated
 *    otherwise; the library allocates nothing. Scratch space is the caller's
 *    `workspace` (size from tt_workspace_bytes).
 *  - Calls are asynchronous on `stream` (a cudaStream_t, NULL = the legacy
 *    default stream). Nothing synchronises; the caller does.
 *  - Call-level errors come back as tt_status before anything is launched.
 *    Per-request problems are reported in status[b] (bits below); a failed
 *    request yields accepted[b] = 0 and next_token[b] = -1. Kernels never trap.
 *  - Requests are CSR batches: request b owns draft tokens
 *    draft_off[b] .. draft_off[b+1]-1 and target tokens
 *    target_off[b] .. target_off[b+1]-1 (k_b and m_b of them). It owns the draft
 *    logits rows with the same indices (row i is the distribution d_i was drawn
 *    from) and the m_b + 1 target logits rows target_off[b] + b ..
 *    target_off[b+1] + b (row j scores t_{j+1}; the last one is the bonus row).
 *  - All indices in inputs and outputs are 0-based.
 *  - Uniforms: Philox4x64-10 (Salmon et al., SC'11), key (seed, 0), counter
 *    (position j, stream, request_base + b, 0), u = (top 24 bits of word 0) *
 *    2^-24; stream 0 draws the accept uniforms, stream 1 the resampling one.
 */
#ifndef TT_H
#define TT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TT_MAX_K 256          /* longest draft sequence per request */
#define TT_MAX_M 512          /* longest proxy target sequence per request */
#define TT_MAX_TOKEN_BYTES 256 /* longest byte string of one token */

typedef enum {
  TT_OK = 0,
  TT_ERR_INVALID_ARG = 1, /* a NULL required pointer, a bad size or alignment */
  TT_ERR_UNSUPPORTED = 2, /* valid but outside what the kernels handle */
  TT_ERR_CUDA = 3         /* a CUDA launch failed; see tt_last_cuda_error() */
} tt_status;

/* Bits of status[b]. */
#define TT_REQ_OK 0
#define TT_REQ_ID_OUT_OF_RANGE 1 /* a token id / logits column / map entry out of range */
#define TT_REQ_TOO_LONG 2        /* k > min(max_k, TT_MAX_K), m > min(max_m, TT_MAX_M) or a
                                    token longer than TT_MAX_TOKEN_BYTES */
#define TT_REQ_EMPTY 4           /* k == 0 or m == 0 */
#define TT_REQ_BAD_OFFSETS 8     /* CSR offsets decreasing or outside [0, n_draft/n_target] */
#define TT_REQ_NOT_FINITE 16     /* a logits row gave a non-finite normaliser */
#define TT_REQ_TIMEOUT 32        /* a pipeline wait in the row pass gave up (bounded waits);
                                    the step's results are not valid */
#define TT_REQ_INTERNAL 64       /* an internal bounds check in a kernel failed (the access
                                    was skipped); the step's results are not valid */
#define TT_REQ_NO_MATCH 128      /* tt_encode: some position of the decoded draft string is
                                    spelled by no token of the target vocabulary */
#define TT_REQ_INCONSISTENT 256  /* tt_consistency: decode_t(T) != decode_d(D) (Lemma 1) */

#define TT_MAX_ENCODE_BYTES 2048 /* longest decoded draft string tt_encode takes per request */
#define TT_MAX_TOP_K 32          /* largest top-k of the sampling filters */
#define TT_MAX_DPOS_BINS 4096    /* most bins of tt_dpos_hist */
#define TT_MAX_HISTORY 3072      /* longest repetition-penalty history per request */

typedef enum { TT_F32 = 0, TT_BF16 = 1 } tt_dtype;

/* A token byte-string table: token id v spells bytes[offsets[v] .. offsets[v+1]). */
typedef struct {
  const uint8_t* bytes;   /* device, [n_bytes] */
  const int64_t* offsets; /* device, [n_tokens + 1]; a token whose range is not inside
                             [0, n_bytes] is reported as TT_REQ_ID_OUT_OF_RANGE */
  int32_t n_tokens;
  int64_t n_bytes;
} tt_vocab;

/* Row-major logits rows: row r starts at element r * row_stride. data must be
 * 16-byte aligned and row_stride * element size a multiple of 16 bytes. */
typedef struct {
  const void* data; /* device */
  int32_t dtype;    /* tt_dtype */
  int32_t n_cols;   /* V: width of a row (the vocabulary the row scores) */
  int64_t row_stride; /* elements between row starts, >= n_cols */
  int64_t n_rows;   /* rows available at data */
} tt_logits;

typedef struct {
  int32_t window;      /* Sakoe-Chiba half-width w >= 0 (the paper settles on 8,
                          App. K); negative = no band. The band used for a request
                          is max(w, |k - m|) so that (k, m) stays reachable. */
  float temp_draft;    /* T_d > 0: draft rows are softmax(z / T_d) */
  float temp_target;   /* T_t > 0: target rows are softmax(z / T_t) */
  int32_t full_q;      /* 0: one-hot transfer (the paper's); 1: homogeneous
                          vocabularies, residual max(0, p - q) against the full
                          draft row (standard speculative decoding, Alg. 4);
                          needs draft and target rows of the same width */
  uint64_t seed;       /* Philox key */
  uint64_t request_base; /* global index of request 0 in the Philox counter */
  void* const* events; /* host array of 4 cudaEvent_t or NULL: tt_step records
                          them before align, before the row pass, before the
                          decision kernel and after it (profiling only) */
  /* Sampling filters of the paper's generation hyperparameters (App. F), per family,
     after the temperature: keep the top_k largest logits of a row (0 = off,
     at most TT_MAX_TOP_K; among equal logits the smaller column first), then
     keep tokens in decreasing probability while the mass before a token is
     below top_p (top_p >= 1 = off), and renormalise the kept set. Every
     probability of the step is then the filtered one: q_hat, p_hat, the accept
     ratio, the residual and the bonus row; lse is the log-normaliser of each
     target row's kept set. top_p < 1 with top_k = 0 keeps a nucleus over the
     whole row (the shortest prefix, larger logit then smaller column first,
     whose mass reaches top_p); in full-q mode either both families are
     filtered or neither, and no family may be a nucleus one
     (TT_ERR_UNSUPPORTED). */
  int32_t top_k_draft;
  float top_p_draft;
  int32_t top_k_target;
  float top_p_target;
  /* Repetition penalty of the same table, per family (1 = off, else > 0): in
     a row, every column of the request's history (tt_batch hist_*) and of the
     sequence tokens before the row's position (target row j: t_1..t_j; draft
     row i: d_1..d_i) has its logit z replaced by z * theta when z < 0, else by
     z / theta (fp32, once per column), before temperature and the filters.
     A penalized family needs top_k >= 1 (TT_ERR_UNSUPPORTED otherwise, and in
     full-q mode). */
  float rep_penalty_draft;
  float rep_penalty_target;
} tt_params;

typedef struct {
  int32_t B;          /* requests */
  int32_t n_draft;    /* sum of k_b = draft_off[B] */
  int32_t n_target;   /* sum of m_b = target_off[B] */
  int32_t max_k;      /* bound on k_b used to size on-chip buffers (<= TT_MAX_K) */
  int32_t max_m;      /* bound on m_b (<= TT_MAX_M) */
  const int32_t* draft_off;   /* [B+1] */
  const int32_t* draft_ids;   /* [n_draft] ids into the draft vocab table */
  const int32_t* draft_cols;  /* [n_draft] column of d_i in its logits row; NULL = draft_ids */
  const int32_t* target_off;  /* [B+1] */
  const int32_t* target_ids;  /* [n_target] ids into the target vocab table */
  const int32_t* target_cols; /* [n_target] column of t_j in its logits row; NULL = target_ids */
  /* Histories of the repetition penalty (read only when that family's penalty
     is on): request b's earlier tokens as logits columns,
     hist_cols[hist_off[b] .. hist_off[b+1]), at most TT_MAX_HISTORY per request
     (TT_REQ_TOO_LONG beyond); NULL hist_off = empty histories. */
  const int32_t* hist_off_d;  /* [B+1] draft family (draft logits columns) */
  const int32_t* hist_cols_d; /* [n_hist_d] */
  const int32_t* hist_off_t;  /* [B+1] target family (target logits columns) */
  const int32_t* hist_cols_t; /* [n_hist_t] */
  int32_t n_hist_d;           /* hist_off_d[B] (sizes the workspace) */
  int32_t n_hist_t;           /* hist_off_t[B] */
} tt_batch;

/* Outputs of tt_step. accepted, next_token and status are required; the rest
 * may be NULL. */
typedef struct {
  int32_t* accepted;   /* [B] a_b, number of target tokens accepted (0..m_b) */
  int32_t* next_token; /* [B] column sampled from the residual / bonus row */
  int32_t* status;     /* [B] TT_REQ_* bits */
  int32_t* path;       /* [2 * (n_draft + n_target)] (i, j) pairs; request b's
                          path starts at pair draft_off[b] + target_off[b] */
  int32_t* path_len;   /* [B] pairs on the path (<= k_b + m_b - 1) */
  int32_t* cost;       /* [B] C* = accumulated cost of the path, -1 if failed */
  int32_t* map;        /* [n_target] draft index aligned to each target token */
  float* q_hat;        /* [n_target] transferred draft probability q(t_j) */
  float* p_hat;        /* [n_target] target probability p(t_j) */
  float* lse;          /* [n_target + B] natural log-normaliser of every target row */
} tt_step_out;

/* Bytes of scratch the transfer / verify / step calls need for this batch and
 * these row widths, without sampling filters. 256-byte aligned sizes; pass a
 * 256-byte aligned pointer. */
size_t tt_workspace_bytes(const tt_batch* batch, int32_t V_d, int32_t V_t);

/* The same with the sampling filters of `prm` (a filtered family keeps, per
 * row, top_k candidates of 8 bytes per unit of 8 KB of logits -- 2048 fp32
 * or 4096 bf16 columns -- and its kept set of top_k entries of 8 bytes). */
size_t tt_workspace_bytes_for(const tt_batch* batch, int32_t V_d, int32_t V_t,
                              const tt_params* prm);

/* (a) DTW alignment (§4.1, Alg. 1; App. H token distance).
 * Per request: local cost d(i,j) = Levenshtein distance between the byte
 * strings of d_i (in vd) and t_j (in vt), for cells inside the band;
 * C_{0,0} = 0, border and out-of-band cells infinite,
 * C_{i,j} = d(i,j) + min(C_{i-1,j}, C_{i,j-1}, C_{i-1,j-1}); backtrack from
 * (k, m) taking the smallest predecessor, ties broken diagonal, then (i-1, j),
 * then (i, j-1). Writes path/path_len/cost/map/status; map[j] is the largest
 * draft index on the path in column j. Uses batch ids (not cols). Needs no
 * workspace. The on-chip tile of a pair takes one byte per band cell (at most
 * about 145 KB of shared memory at max_k = TT_MAX_K, max_m = TT_MAX_M with no
 * band), so every allowed size fits; TT_ERR_UNSUPPORTED would report one that
 * did not. */
tt_status tt_align(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                   const tt_params* prm, int32_t* path, int32_t* path_len, int32_t* cost,
                   int32_t* map, int32_t* status, void* stream);

/* (b) Transfer (Alg. 2 MapProbabilities, App. A.2, Limitations).
 * q_hat[j] = softmax(draft row map[j] / T_d) at column draft_cols[map[j]],
 * or draft_probs[draft_off[b] + map[j]] when draft_probs (fp32 [n_draft],
 * device) is not NULL, in which case `draft` may be NULL. Writes q_hat and
 * status. */
tt_status tt_transfer(const tt_batch* batch, const int32_t* map, const tt_logits* draft,
                      const float* draft_probs, const tt_params* prm, void* workspace,
                      size_t workspace_bytes, float* q_hat, int32_t* status, void* stream);

/* (c) Verification (§4.2, Alg. 2 accept loop, Alg. 4 residual).
 * Reads the m_b + 1 target rows of every request once. p_hat[j] =
 * softmax(target row j / T_t) at target_cols[j]; accept while
 * u_j < min(1, p_hat[j] / q_hat[j]) (q_hat = 0 accepts when p_hat > 0);
 * a_b = accepted count; next token from row a_b: residual max(0, p - q)
 * (one-hot q = q_hat e_{t}, or the full draft row map[a_b] when full_q), or
 * the bonus row itself when a_b = m_b; inverse CDF in column order, smallest x
 * whose running mass exceeds u' * Z. `draft` and `map` are read only when
 * full_q. p_hat and lse may be NULL. */
tt_status tt_verify(const tt_batch* batch, const float* q_hat, const tt_logits* target,
                    const tt_logits* draft, const int32_t* map, const tt_params* prm,
                    void* workspace, size_t workspace_bytes, int32_t* accepted,
                    int32_t* next_token, float* p_hat, float* lse, int32_t* status,
                    void* stream);

/* (a)+(b)+(c) fused: align, one streaming pass over the needed draft rows and
 * all target rows, then the per-request decision, as three kernels on
 * `stream`. Same results as tt_align -> tt_transfer -> tt_verify. */
tt_status tt_step(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                  const tt_logits* draft, const float* draft_probs, const tt_logits* target,
                  const tt_params* prm, void* workspace, size_t workspace_bytes,
                  const tt_step_out* out, void* stream);

/* Device scratch, in bytes, that the library keeps for tt_step_noalloc. */
#define TT_NOALLOC_SCRATCH_BYTES (16u << 20)

/* tt_step for callers that cannot allocate device memory. (The paper has no
 * counterpart: this is a deployment aid of this library.)
 * Some callers cannot call cudaMalloc or any other allocating routine where they
 * run a verification step: runtimes whose device memory is owned by one arena
 * that must not be bypassed, serving loops that must not stall on the
 * allocator (cudaMalloc can synchronise the device), or foreign-language hosts
 * that only hand over input and output buffers. Such callers cannot provide the
 * `workspace` of tt_step. This entry point takes the same arguments minus the
 * workspace and uses a fixed scratch array of TT_NOALLOC_SCRATCH_BYTES (16 MiB)
 * compiled into the library: every GPU that loads the library holds those
 * 16 MiB until the process exits. It allocates nothing.
 *  - Every argument check of tt_step runs first, on the host; a refused call
 *    queues nothing on `stream`. Batches that need more scratch than the
 *    array holds (tt_workspace_bytes_for with these params) are then refused
 *    with TT_ERR_UNSUPPORTED; the five workloads the library is measured on
 *    all fit.
 *  - The scratch used is the current device's (devices 0..63; others get
 *    TT_ERR_UNSUPPORTED): `stream` must belong to the current device. The
 *    first call on each device looks up the array's device address there
 *    (cudaGetSymbolAddress, once per device even with several host threads);
 *    make that first call before any stream capture.
 *  - Every call on a device shares the one array, which keeps the last call's
 *    contents; nothing in it needs to start at zero (every value is written
 *    before it is read, and the row pass's error report is tagged with the
 *    call it belongs to). Calls whose work overlaps on the GPU (two streams,
 *    or two host threads) race on the array: order them.
 * Results equal tt_step's for the same arguments. */
tt_status tt_step_noalloc(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                          const tt_logits* draft, const float* draft_probs,
                          const tt_logits* target, const tt_params* prm,
                          const tt_step_out* out, void* stream);

/* ------------------------------------------------------------------------
 * Re-encoding and its checks (§4.2; App. A.1, Lemma 1; §4.1 and App. K).
 * ---------------------------------------------------------------------- */

/* Size of the re-encoding index of a vocabulary with n_tokens tokens and
 * n_bytes bytes of strings (an open-addressing table of every prefix of every
 * token, 16 bytes per slot, at most half full). */
size_t tt_vocab_index_bytes(int32_t n_tokens, int64_t n_bytes);

/* Builds the re-encoding index of a target vocabulary. HOST pointers in and
 * out: `bytes`/`offsets` as in tt_vocab, `index` a host buffer of
 * tt_vocab_index_bytes() bytes; the caller copies it to the device once (it
 * is position-independent) and passes the device copy to tt_encode. Among
 * tokens with equal strings the smallest id is kept; empty tokens are left
 * out. TT_ERR_UNSUPPORTED for a token longer than TT_MAX_TOKEN_BYTES, or in
 * the (never observed) event of two different prefixes longer than 8 bytes
 * with equal 64-bit fingerprints. Synchronous, deterministic. */
tt_status tt_vocab_index_build(const uint8_t* bytes, const int64_t* offsets, int32_t n_tokens,
                               void* index, size_t index_bytes);

/* Scratch of tt_encode for B requests of at most max_m target tokens. */
size_t tt_encode_workspace_bytes(int32_t B, int32_t max_m);

/* T_b = encode_t(decode_d(D_b)) for every request (§4.2, App. A.1): the draft
 * tokens' byte strings (in vd) concatenated, then greedy longest match over
 * the target vocabulary (vt, with its index vt_index from
 * tt_vocab_index_build): at each position the longest target token spelling
 * the next bytes, the smallest id among equal strings. This is the tokenizer
 * of the synthetic workloads; a learned tokenizer's merges are not modelled.
 * Inputs: B, n_draft (= draft_off[B]), draft_off [B+1], draft_ids [n_draft]
 * (device). Outputs (device):
 * target_off [B+1], target_ids [capacity], status [B]. Status bits: BAD_OFFSETS,
 * ID_OUT_OF_RANGE (a draft id), EMPTY (k = 0), TOO_LONG (decoded string longer
 * than TT_MAX_ENCODE_BYTES, more than max_m tokens, or the request's tokens
 * would end past `capacity` counting every earlier request's tokens, written
 * or not), NO_MATCH. A failed request writes no tokens:
 * target_off[b+1] = target_off[b] + (tokens written for b). */
tt_status tt_encode(int32_t B, int32_t n_draft, const int32_t* draft_off, const int32_t* draft_ids,
                    const tt_vocab* vd, const tt_vocab* vt, const void* vt_index,
                    int32_t max_m, int32_t capacity, int32_t* target_off,
                    int32_t* target_ids, int32_t* status, void* workspace,
                    size_t workspace_bytes, void* stream);

/* Lemma 1 (App. A.1) as a check on any (D, T), e.g. a T re-encoded by the
 * caller's own tokenizer: status[b] = 0 when the bytes of T_b are those of
 * D_b, TT_REQ_INCONSISTENT when they differ, BAD_OFFSETS / ID_OUT_OF_RANGE /
 * TOO_LONG (k > max_k or m > max_m) otherwise. Uses ids, not cols. */
tt_status tt_consistency(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                         int32_t* status, void* stream);

/* Delta-pos (§4.1, App. K), the position deviation of DTW-matched tokens,
 * counted into hist[min(delta, n_bins - 1)] (int64, device, ADDED to: zero it
 * before the first call; many steps can be accumulated). mode 0: delta = |i - j|
 * for every pair on each request's path (tt_align's path / path_len); mode 1:
 * delta = |map[j] - j| for every target position. Requests with path_len[b] <= 0
 * add nothing. n_bins in [1, TT_MAX_DPOS_BINS]. The paper chooses w where the
 * cumulative distribution of delta (taken with no band) reaches 0.9. */
tt_status tt_dpos_hist(const tt_batch* batch, const int32_t* path, const int32_t* path_len,
                       const int32_t* map, int32_t mode, int32_t n_bins, int64_t* hist,
                       void* stream);

/* ---------------------------------------------------------------------------
 * Vocabulary-sharded verification, emulated on one GPU.
 *
 * A tensor-parallel target model leaves each rank with a column slice of every
 * target logits row. The verification step (c) then needs one exchange: every
 * rank reduces its slice of each row to a summary (its max and sum of
 * exponentials with the scored token left out, and the scored token's logit
 * if the rank owns it); the summaries of all ranks are gathered; the merged
 * normalisers give p(t_j) and the accept test exactly as in tt_verify; the
 * residual row's mass per shard picks the shard that holds the drawn point,
 * and only that shard's slice is read again to find the column.
 * tt_verify_sharded runs that protocol with the S shards as S logits arrays on
 * one device: each shard's slice is reduced by its own row pass, and the
 * gathered summaries are a device buffer in the layout an all-gather would
 * produce ([S][n_target + B] records of 16 bytes). Results equal tt_verify's
 * on the concatenated rows up to rounding (same uniforms, same column order).
 * One-hot transfer only, no sampling filters (TT_ERR_UNSUPPORTED otherwise).
 */
#define TT_MAX_SHARDS 8

typedef struct {
  int32_t S;                /* shards, 1 .. TT_MAX_SHARDS */
  const tt_logits* shards;  /* HOST array of S descriptors; shard s holds columns
                               col0[s] .. col0[s] + shards[s].n_cols - 1 of every
                               target row (n_target + B rows, as in tt_verify) */
  const int32_t* col0;      /* HOST array of S first columns: col0[0] = 0 and the
                               shards tile the row in order without gaps */
} tt_shards;

/* Scratch bytes of tt_verify_sharded (256-byte aligned size). */
size_t tt_sharded_workspace_bytes(const tt_batch* batch, const tt_shards* target);

/* Verification over sharded target rows. q_hat [n_target] as for tt_verify;
 * accepted / next_token / status [B], p_hat [n_target] and lse [n_target + B]
 * (both optional) as for tt_verify; next_token is a column of the whole row.
 * summaries (optional, [S * (n_target + B) * 4] floats) receives the gathered
 * per-shard records (max and sum of 2^(z * log2(e) / T - max) over the shard's
 * columns without the scored one, that sum's low word, and the scored
 * token's scaled logit or NaN), for inspection. */
tt_status tt_verify_sharded(const tt_batch* batch, const float* q_hat, const tt_shards* target,
                            const tt_params* prm, void* workspace, size_t workspace_bytes,
                            int32_t* accepted, int32_t* next_token, float* p_hat, float* lse,
                            float* summaries, int32_t* status, void* stream);

/* Static text for a tt_status. */
const char* tt_status_string(tt_status s);

/* cudaError_t of the last failed launch in this process (0 if none). */
int32_t tt_last_cuda_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t tt_version(void);

#ifdef __cplusplus
}
#endif
#endif /* TT_H */
