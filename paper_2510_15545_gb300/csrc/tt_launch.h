// tt_launch.h -- kernel argument blocks and launchers (internal to libtt).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/tt.h"

namespace tt {

struct Partial;

constexpr int kAlignWarpsMax = 4;             // sequence pairs per align CTA
constexpr int kAlignSmemMax = 200 * 1024;     // dynamic shared memory cap of one align CTA
constexpr int kMaxChunksPerRow = 256;         // rows up to 256 * 8192 = 2,097,152 columns

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
  const int32_t* target_cols;  // with excl: columns of the scored target tokens
  int V_t;                     // width of the target rows (excl only)
  int32_t* excl;               // [n_target + B] scored column of each target row, -1 if none (may be NULL)
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
  Partial* part;
  const uint8_t* need;  // rows to visit (NULL = all)
};

struct RowPassArgs {
  RowSet d, t;
  int64_t items_d, items_t;  // rows * chunks of each family (0 = family absent)
  const int32_t* excl;       // [target rows]: column left out of the sum, -1 = none
};

struct DecideArgs {
  int B, n_draft, n_target, max_m, full_q, mode_transfer_only;
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
  uint64_t seed, request_base;
  int32_t* accepted;
  int32_t* next_token;
  int32_t* status;
  float* q_hat_out;
  float* p_hat;
  float* lse;
};

struct PrepArgs {
  int B, n_draft, n_target, V_t;
  const int32_t* draft_off;
  const int32_t* target_off;
  const int32_t* target_cols;
  const int32_t* map;
  uint8_t* need;   // written from map when not NULL
  int32_t* excl;   // written from target_cols when not NULL
};

size_t align_smem_per_warp(int max_k, int max_m, int tile_w);
int align_tile_width(int max_k, int max_m, int window);
cudaError_t launch_align(const AlignArgs& args, cudaStream_t stream);
cudaError_t launch_rowpass(const RowPassArgs& args, int dt_d, int dt_t, cudaStream_t stream,
                           int sm_count);
cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream);
cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream);

}  // namespace tt
