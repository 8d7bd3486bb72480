// tt_launch.h -- kernel argument blocks and launchers (internal to libtt).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "tt.h"

namespace tt {

struct Partial;

constexpr int kAlignWarpsMax = 8;             // warps (pairs at a time) per align CTA
constexpr int kAlignWarpsStep = 4;            // the same inside tt_step, beside the row pass
constexpr int kAlignSmemMax = 200 * 1024;     // dynamic shared memory cap of one align CTA
constexpr int kMaxChunksPerRow = 1024;        // rows up to 1024 * 2048 = 2,097,152 columns

struct AlignArgs {
  int B, n_draft, n_target, max_k, max_m, window;
  const int32_t* draft_off;
  const int32_t* draft_ids;
  const int32_t* target_off;
  const int32_t* target_ids;
  tt_vocab vd, vt;
  int32_t* path;
  int32_t* path_len;
  int32_t* cost;
  int32_t* map;
  int32_t* status;
  uint8_t* need;               // needed draft rows (may be NULL)
  unsigned long long* work;    // row-pass work counters to zero (may be NULL)
  const int32_t* target_cols;  // scored column of each target position
  int32_t* excl;               // [n_target + B] written: scored column of each target row
                               // (-1 for the bonus row), may be NULL
  int warps_per_block, tile_w;
  size_t smem_per_warp;
};

// One family of logits rows seen by the row pass.
struct RowSet {
  const char* data;
  int64_t stride_bytes;
  int V;
  int nch;
  float scale;  // log2(e) / T
  int64_t n_rows;
  Partial* part;
  const uint8_t* need;  // rows to visit (NULL = all)
  int top_k;            // > 0: filtered rows, the row pass writes top-k lists to cand
  Cand* cand;           // [n_rows * nlist * cand_stride(top_k)]: one list per row unit
  int nlist;            // units (8 KB stages: 2048 fp32 or 4096 bf16 columns) per row
  int nucleus;          // 1: top-p without top-k (top_k = 0): the row pass writes the
                        // compensated partials of all its columns; the nucleus
                        // kernel finds each row's kept set
  // Repetition penalty (top-k families only; pen = NULL: none): the row pass
  // leaves each request's penalized columns out of its unit lists, and the
  // kept-set kernel adds them back with the row's own (penalized or raw) value.
  const PenEntry* pen;    // sorted penalized columns of request b at pbase[b] (pcnt[b])
  const int32_t* pbase;
  const int32_t* pcnt;
  const int32_t* pstart;  // [B * (nch + 1)]: first entry of each row unit, then pcnt
  float penalty;          // theta
  int unit_cols;          // columns per row unit (2048 fp32, 4096 bf16)
};

struct RowPassArgs {
  RowSet d, t;
  int64_t rows_d, rows_t;    // rows of each family to stream (0 = family absent)
  const int32_t* excl;       // [target rows] column left out of the sum, or NULL: found
                             // from target_off / target_cols
  int B, n_target, n_draft;
  const int32_t* target_off;
  const int32_t* target_cols;
  const int32_t* draft_off;  // to find a penalized draft row's request
  int32_t* err;              // err[0] = epoch of a failed call, err[1] = its TT_REQ_* bits
  int32_t epoch;             // identifies this call
  const int32_t* excl_late;  // as excl, but written by the grid this one depends on: read
                             // only after the grid-dependency wait (may be NULL)
  // Work counter for the items past each CTA's fixed share, zeroed by the grid
  // this one depends on and read only after the grid-dependency wait; NULL:
  // every item belongs to a fixed share.
  unsigned long long* work;
  int32_t pre_eighths;       // with work: eighths of the target items streamed in fixed
                             // blocks before the grid-dependency wait (1..7)
  int32_t stall_stage;       // test hook (-1 = off): in CTA 0 the stage consumed at
                             // consumer step stall_stage is never freed, so the
                             // bounded waits run out
  uint64_t wait_ns;          // limit of every pipeline wait (set by launch_rowpass: 2 s)
};

struct DecideArgs {
  int B, n_draft, n_target, max_k, max_m, full_q, mode_transfer_only;
  const int32_t* draft_off;
  const int32_t* draft_cols;
  const int32_t* target_off;
  const int32_t* target_cols;
  const int32_t* map;
  const float* q_hat_in;     // given q_hat (verify) or NULL (computed here)
  const float* draft_probs;  // given draft probabilities or NULL
  RowSet d, t;
  int dt_d, dt_t;
  const int32_t* status_in;  // status of an earlier stage (align) or NULL
  int32_t* err;              // row-pass error words (NULL when no row pass ran)
  int32_t epoch;
  uint64_t seed, request_base;
  int32_t* accepted;
  int32_t* next_token;
  int32_t* status;
  float* q_hat_out;
  float* p_hat;
  float* lse;
  int warm_ctas;  // CTAs b < warm_ctas run a warming pass before the wait (see decide.cu)
  int sm_count;   // SMs of the device (sizes the decision kernel's CTAs)
  float top_p_d, top_p_t;    // top-p of filtered families (d.top_k / t.top_k > 0)
  const int32_t* status_q;   // status of the kernel that produced q_hat_in, or NULL
  const Cand* kept_d;        // kept sets of filtered families (written by the kept kernel)
  const Cand* kept_t;
  const KeptHead* head_d;
  const KeptHead* head_t;
  const float* um_d;         // per-chunk kept masses of nucleus families
  const float* um_t;
  const int32_t* status_p;   // problems of the repetition-penalty histories, or NULL
};

// The kept-set stage of filtered families: one warp per row merges the row's
// unit lists into its top-k and applies temperature and top-p.
struct KeptArgs {
  RowSet d, t;             // families with top_k > 0 (kept_kernel) or nucleus (nucleus_kernel)
                           // are done, the others skipped
  int64_t rows_d, rows_t;  // rows of each family (draft rows with d.need[row] == 0 skipped)
  float top_p_d, top_p_t;
  Cand* kept_d;
  Cand* kept_t;
  KeptHead* head_d;
  KeptHead* head_t;
  float* um_d;             // nucleus families: kept probability mass per chunk
  float* um_t;
  int dt_d, dt_t;          // logits types (nucleus rows are read again)
  int B, n_target;         // the batch, to find a nucleus target row's scored column
  const int32_t* target_off;
  const int32_t* target_cols;
  const int32_t* draft_off;  // and a penalized draft row's request
  int n_draft;
};

// The repetition penalty's per-request sets (pen.cu): for each penalized
// family, every request's history and sequence columns sorted and made unique
// (with the first sequence position of each), and the start of each row unit.
struct PenArgs {
  int B;
  int on_d, on_t;
  int V_d, V_t, nch_d, nch_t, unit_d, unit_t, nlist_d, nlist_t;
  int n_draft, n_target, n_hist_d, n_hist_t;
  const int32_t* hist_off_d;
  const int32_t* hist_cols_d;
  const int32_t* hist_off_t;
  const int32_t* hist_cols_t;
  const int32_t* draft_off;
  const int32_t* draft_cols;
  const int32_t* target_off;
  const int32_t* target_cols;
  PenEntry* pen_d;
  int32_t* pbase_d;
  int32_t* pcnt_d;
  int32_t* pstart_d;
  PenEntry* pen_t;
  int32_t* pbase_t;
  int32_t* pcnt_t;
  int32_t* pstart_t;
  int32_t* pstatus;
};

struct PrepArgs {
  int B, n_draft, n_target;
  const int32_t* draft_off;
  const int32_t* target_off;
  const int32_t* map;
  uint8_t* need;   // needed-draft-row flags, written from map
  unsigned long long* work;  // row-pass work counter to zero (may be NULL)
};

size_t align_smem_per_warp(int max_k, int max_m, int tile_w);
int align_tile_width(int max_k, int max_m, int window);
cudaError_t launch_align(const AlignArgs& args, cudaStream_t stream);
cudaError_t launch_rowpass(const RowPassArgs& args, int dt_d, int dt_t, cudaStream_t stream,
                           int sm_count, bool pdl);
cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream, bool pdl);
cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream);

// Filtered families (filter.cu): the kept sets of the filtered rows from their
// top-k lists, then q_hat of every target position from the kept sets of the
// mapped draft rows, and the decision over filtered target rows
// (args.t.top_k > 0) with q_hat_in given.
cudaError_t launch_kept(const KeptArgs& args, cudaStream_t stream, int sm_count, bool pdl);
// Nucleus families (top-p without top-k, App. F): the exact kept set of every
// nucleus row from its logits and the row pass's partials, and the decision
// over nucleus target rows.
cudaError_t launch_nucleus(const KeptArgs& args, cudaStream_t stream, int sm_count, bool pdl);
cudaError_t launch_decide_nucleus(const DecideArgs& args, cudaStream_t stream, bool pdl);
cudaError_t launch_pen_prep(const PenArgs& args, cudaStream_t stream);
cudaError_t launch_filter_q(const DecideArgs& args, cudaStream_t stream, bool pdl);
cudaError_t launch_decide_filtered(const DecideArgs& args, cudaStream_t stream, bool pdl);

// Loads every kernel of the library on the current device and sets its launch
// attributes, so that no module is loaded lazily inside a dependent-launch chain.
cudaError_t preload_align();
cudaError_t preload_rowpass();
cudaError_t preload_decide();
cudaError_t preload_filter();
cudaError_t preload_nucleus();
cudaError_t preload_pen();

// Records a failed CUDA call for tt_last_cuda_error() and returns TT_ERR_CUDA.
tt_status record_cuda_error(cudaError_t e);

// Every argument check of tt_step, on the host only (nothing is queued on a
// stream): TT_OK and the workspace bytes the step needs (0 for an empty batch),
// or the status tt_step would return for these arguments.
tt_status step_check(const tt_batch* batch, const tt_vocab* vd, const tt_vocab* vt,
                     const tt_logits* draft, const float* draft_probs, const tt_logits* target,
                     const tt_params* prm, const tt_step_out* out, size_t* need);

}  // namespace tt
