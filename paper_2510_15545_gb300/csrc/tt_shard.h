// tt_shard.h -- argument blocks and launchers of the vocabulary-sharded
// verification (shard.cu), emulated on one GPU (internal to libtt).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "tt.h"

namespace tt {

struct Partial;

struct ShardDesc {
  const char* data;      // the shard's logits (device)
  int64_t stride_bytes;  // between rows
  int32_t V;             // columns of the slice
  int32_t col0;          // first column of the whole row
  int32_t nch;           // 2048-column chunks of the slice
  int32_t dtype;
  Partial* part;         // [rows * nch] chunk partials of the slice
};

// One gathered record: shard s, row r.
struct ShardRec {
  float m;       // max of s_x = z_x * log2(e) / T over the slice without the scored column
  float s_hi;    // sum of 2^(s_x - m) over the same columns, as hi + lo
  float s_lo;
  float st;      // s of the scored column if this shard owns it, else NaN
};
static_assert(sizeof(ShardRec) == 16, "records are 4 floats");

struct ShardArgs {
  int B, n_target, S, V, max_m;
  int64_t rows;  // n_target + B
  const int32_t* target_off;
  const int32_t* target_cols;
  ShardDesc sh[TT_MAX_SHARDS];
  int32_t* excl;             // [S * rows] scored column within each shard, or -1
  ShardRec* rec;             // [S * rows]
  unsigned long long* work;  // S row-pass work counter blocks (zeroed by shard_excl_kernel)
  float scale;               // log2(e) / T_t
  const float* q_hat;
  uint64_t seed, request_base;
  const int32_t* err;        // row-pass error words
  int32_t epoch;
  int32_t* accepted;
  int32_t* next_token;
  int32_t* status;
  float* p_hat;
  float* lse;
};

struct ShardWorkspace {
  Partial* part[TT_MAX_SHARDS];
  int32_t* excl;
  ShardRec* rec;
  unsigned long long* work;  // S blocks of kWorkBlockBytes
  int32_t* err;
  size_t bytes;
};

// Workspace of tt_verify_sharded; nch[s] = chunks of shard s.
ShardWorkspace shard_layout(void* base, int64_t rows, int S, const int32_t* nch);
cudaError_t launch_shard_excl(const ShardArgs& args, cudaStream_t stream);
cudaError_t launch_shard_summary(const ShardArgs& args, cudaStream_t stream, int sm_count);
cudaError_t launch_decide_sharded(const ShardArgs& args, cudaStream_t stream);

cudaError_t preload_shard();

}  // namespace tt
