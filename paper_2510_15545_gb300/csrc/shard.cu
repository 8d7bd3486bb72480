// shard.cu -- verification (§4.2, Alg. 2 / Alg. 4, one-hot transfer) over
// target rows split by columns into S shards, as a tensor-parallel target
// model leaves them, emulated on one GPU.
//
// Per shard (what one rank does with its slice): a row pass over the slice
// gives chunk partials with the scored token left out; shard_summary_kernel
// reduces them to one record per row (max, sum of 2^(s - max) as an fp64 pair
// of floats, the owned scored token's scaled logit or NaN). The records of all
// shards are the exchange (an all-gather across ranks; here a device buffer in
// that layout). decide_sharded_kernel merges them (split-lse), runs the accept
// test with the same Philox uniforms as the unsharded path, and samples the
// residual (or the bonus row) by inverse CDF in column order at three levels:
// the shard from the merged records, the chunk within that shard from its
// partials, and the column from one re-read chunk of that shard's slice.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>

#include "tt_device.cuh"
#include "tt_launch.h"
#include "tt_shard.h"

namespace tt {

namespace {

constexpr int kShThreads = 256;

// Column of the whole row scored by target row r (-1: a bonus row, or an
// entry the decision reports as out of range): request b owns rows
// target_off[b] + b .. target_off[b+1] + b.
__device__ int scored_column(const ShardArgs& a, int64_t r) {
  if (a.B <= 0) return -1;
  int lo = 0, hi = a.B - 1;
  while (lo < hi) {  // largest b with target_off[b] + b <= r
    const int mid = (lo + hi + 1) >> 1;
    if (int64_t(a.target_off[mid]) + mid <= r) lo = mid;
    else hi = mid - 1;
  }
  const int b = lo;
  const int t0 = a.target_off[b], t1 = a.target_off[b + 1];
  if (t0 < 0 || t1 < t0 || t1 > a.n_target) return -1;
  const int64_t j = r - (int64_t(t0) + b);
  if (j < 0 || j >= t1 - t0) return -1;
  const int c = a.target_cols[t0 + j];
  return (c >= 0 && c < a.V) ? c : -1;
}

// Each shard's own scored column of every target row; zeroes the row passes'
// work counters and the error words.
__global__ void shard_excl_kernel(ShardArgs a, int32_t* err) {
  const int64_t i0 = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i0 < int64_t(kWorkShards) * kWorkStride * a.S) a.work[i0] = 0ull;
  if (i0 < 2) err[i0] = 0;
  for (int64_t r = i0; r < a.rows; r += int64_t(gridDim.x) * blockDim.x) {
    const int c = scored_column(a, r);
    for (int s = 0; s < a.S; ++s) {
      const int x = c - a.sh[s].col0;
      a.excl[s * a.rows + r] = (c >= 0 && x >= 0 && x < a.sh[s].V) ? x : -1;
    }
  }
}

// One warp per (shard, row): the shard's record from its chunk partials.
__global__ void shard_summary_kernel(ShardArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t w0 = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t stride = (int64_t(gridDim.x) * blockDim.x) >> 5;
  for (int64_t w = w0; w < a.S * a.rows; w += stride) {
    const int s = int(w / a.rows);
    const int64_t r = w - int64_t(s) * a.rows;
    const ShardDesc& d = a.sh[s];
    float M;
    double Ssum;
    row_norm_warp(d.part + r * d.nch, d.nch, lane, M, Ssum);
    if (lane == 0) {
      const int x = a.excl[s * a.rows + r];
      float st = __int_as_float(0x7fffffff);
      if (x >= 0) {
        const char* row = d.data + r * d.stride_bytes;
        const float z = d.dtype == TT_F32 ? load_logit<TT_F32>(row, x) : load_logit<TT_BF16>(row, x);
        st = z * a.scale;
      }
      const float hi = float(Ssum);
      a.rec[w] = ShardRec{M, hi, float(Ssum - double(hi)), st};
    }
  }
}

// 2^(x - M) in fp64 for the per-row quantities (0 for -inf or NaN x).
__device__ __forceinline__ double pow2_rel(float x, float M) {
  return (x > -INFINITY) ? exp2_split(double(x) - double(M)) : 0.0;
}

// Inclusive prefix over the warp's lanes in fp64.
__device__ __forceinline__ double warp_scan_d(double v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double x = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += x;
  }
  return v;
}

// One CTA per request: merge the gathered records of the request's m + 1
// target rows (split-lse), accept test, residual or bonus draw.
__global__ void __launch_bounds__(kShThreads) decide_sharded_kernel(ShardArgs a) {
  constexpr int kWarps = kShThreads / 32;
  constexpr int kPer = kChunk / kShThreads;  // columns per thread in the fine level
  __shared__ float s_p[TT_MAX_M];
  __shared__ double s_wsum[kWarps];
  __shared__ int s_acc, s_bad, s_shard, s_chunk, s_hit, s_last;
  __shared__ double s_theta, s_tterm;
  __shared__ float s_M;
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int st = 0, t0 = 0, m = 0;
  if (!csr_ok(a.target_off, b, a.n_target)) {
    st = TT_REQ_BAD_OFFSETS;
  } else {
    t0 = a.target_off[b];
    m = a.target_off[b + 1] - t0;
    if (m == 0) st |= TT_REQ_EMPTY;
    if (m > a.max_m || m > TT_MAX_M) st |= TT_REQ_TOO_LONG;
  }
  int bad = 0;
  if (st == 0)
    for (int j = tid; j < m; j += kShThreads) {
      const int c = a.target_cols[t0 + j];
      if (c < 0 || c >= a.V) bad = 1;
    }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st == 0 && a.err && a.err[0] == a.epoch) st = a.err[1];  // a row pass failed
  if (st != 0) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = st;
    }
    return;
  }
  if (tid == 0) {
    s_acc = m;
    s_bad = 0;
    s_hit = 0x7fffffff;
    s_last = -1;
  }
  __syncthreads();
  const ShardRec none = {-INFINITY, 0.f, 0.f, __int_as_float(0x7fffffff)};
  // the merge: lane s holds shard s's record of the row
  for (int j = warp; j <= m; j += kWarps) {
    const int64_t row = int64_t(t0) + b + j;
    const ShardRec R = lane < a.S ? a.rec[lane * a.rows + row] : none;
    const float M = warp_max_f(fmaxf(R.m, R.st));  // fmaxf skips the NaN of a non-owner
    double z = 0.0, pt = 0.0;
    if (M > -INFINITY && M < INFINITY) {
      z = (double(R.s_hi) + double(R.s_lo)) * pow2_rel(R.m, M);
      pt = pow2_rel(R.st, M);
    }
    z = warp_sum_d(z + pt);
    pt = warp_sum_d(pt);  // the one owner's term
    const bool ok = M > -INFINITY && M < INFINITY && z > 0.0 && z < INFINITY;
    if (lane == 0) {
      if (!ok) s_bad = 1;
      const float p = ok ? float(pt / z) : 0.f;
      if (j < m) {
        s_p[j] = p;
        if (a.p_hat) a.p_hat[t0 + j] = p;
      }
      if (a.lse) a.lse[row] = ok ? float((double(M) + log2_split(z)) * 0.6931471805599453) : NAN;
    }
  }
  __syncthreads();
  if (s_bad) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = TT_REQ_NOT_FINITE;
    }
    return;
  }
  // accept while u_j q_j < p_j (u < 1 exactly)
  const uint64_t req = a.request_base + uint64_t(b);
  for (int j = tid; j < m; j += kShThreads) {
    const float u = float(philox_uniform(a.seed, uint64_t(j), 0, req));
    if (!(u * a.q_hat[t0 + j] < s_p[j])) atomicMin(&s_acc, j);
  }
  __syncthreads();
  const int acc = s_acc;
  const int64_t row = int64_t(t0) + b + acc;
  // residual row acc (or the bonus row): shard, then chunk, in warp 0
  if (warp == 0) {
    const ShardRec R = lane < a.S ? a.rec[lane * a.rows + row] : none;
    const float M = warp_max_f(fmaxf(R.m, R.st));
    const double base = (double(R.s_hi) + double(R.s_lo)) * pow2_rel(R.m, M);
    const double pt = pow2_rel(R.st, M);  // nonzero on the owner only (none on a bonus row)
    const double Z = warp_sum_d(base + pt);
    const double q = acc < m ? double(a.q_hat[t0 + acc]) : 0.0;
    // what the one-hot residual max(0, p - q e_t) leaves at t, times Z
    double tterm = fmax(0.0, pt - q * Z);
    double mass = base + tterm;
    if (!(warp_sum_d(mass) > 0.0)) {  // nothing left: the row itself
      tterm = pt;
      mass = base + pt;
    }
    if (lane >= a.S) mass = 0.0;
    const double incl = warp_scan_d(mass, lane);
    const double tot = __shfl_sync(0xffffffffu, incl, 31);
    const double theta = philox_uniform(a.seed, uint64_t(acc), 1, req) * tot;
    const double before = incl - mass;
    // the first shard whose running mass passes theta; rounding past the end:
    // the last shard with mass
    const unsigned hm = __ballot_sync(0xffffffffu, mass > 0.0 && theta >= before && theta < incl);
    const unsigned pm = __ballot_sync(0xffffffffu, mass > 0.0);
    const int sh = hm ? __ffs(hm) - 1 : (pm ? 31 - __clz(pm) : -1);
    if (sh >= 0) {
      const double th1 = fmin(fmax(theta - __shfl_sync(0xffffffffu, before, sh), 0.0),
                              __shfl_sync(0xffffffffu, mass, sh));
      const double tt = __shfl_sync(0xffffffffu, R.st == R.st ? tterm : 0.0, sh);
      // chunk level within shard sh: its partials, the scored column's term added
      const ShardDesc& d = a.sh[sh];
      const Partial* pp = d.part + row * d.nch;
      const int xs = a.excl[sh * a.rows + row];
      const int tch = xs >= 0 ? xs / kChunk : -1;
      double carry = 0.0;
      int chunk = -1, lastc = -1;
      double th2 = 0.0;
      for (int c0 = 0; c0 < d.nch && chunk < 0; c0 += 32) {
        const int c = c0 + lane;
        double cm = 0.0;
        if (c < d.nch) {
          const Partial P = pp[c];
          cm = double(P.s) * pow2_rel(P.m, M) + (c == tch ? tt : 0.0);
        }
        const double ci = warp_scan_d(cm, lane) + carry;
        const double cb = ci - cm;
        const unsigned h = __ballot_sync(0xffffffffu, cm > 0.0 && th1 >= cb && th1 < ci);
        const unsigned pz = __ballot_sync(0xffffffffu, cm > 0.0);
        if (pz) lastc = c0 + 31 - __clz(pz);
        if (h) {
          chunk = c0 + __ffs(h) - 1;
          th2 = th1 - __shfl_sync(0xffffffffu, cb, __ffs(h) - 1);
        }
        carry = __shfl_sync(0xffffffffu, ci, 31);
      }
      if (chunk < 0 && lastc >= 0) {  // rounding past the end: the last chunk with mass
        chunk = lastc;
        th2 = INFINITY;
      }
      if (lane == 0) {
        s_shard = sh;
        s_chunk = chunk;
        s_theta = th2;
        s_tterm = tt;
        s_M = M;
      }
    } else if (lane == 0) {
      s_shard = -1;
      s_chunk = -1;
    }
  }
  __syncthreads();
  const int sh = s_shard, chunk = s_chunk;
  int pick = -1;
  if (sh >= 0 && chunk >= 0) {
    // column level: the whole CTA re-reads the chunk of shard sh
    const ShardDesc& d = a.sh[sh];
    const float M = s_M;
    const double th2 = s_theta, tt = s_tterm;
    const int xs = a.excl[sh * a.rows + row];
    const int c0 = chunk * kChunk + tid * kPer;
    const char* rp = d.data + row * d.stride_bytes;
    double mine = 0.0;
    double mx[kPer];
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      const int x = c0 + k;
      double w = 0.0;
      if (x < d.V) {
        if (x == xs) {
          w = tt;
        } else {
          const float z = d.dtype == TT_F32 ? load_logit<TT_F32>(rp, x) : load_logit<TT_BF16>(rp, x);
          w = pow2_rel(z * a.scale, M);
        }
      }
      mx[k] = w;
      mine += w;
    }
    const double wi = warp_scan_d(mine, lane);
    if (lane == 31) s_wsum[warp] = wi;
    __syncthreads();
    double off = 0.0;
    for (int w = 0; w < warp; ++w) off += s_wsum[w];
    double run = off + wi - mine;  // mass before this thread's first column
    int last = -1;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      if (mx[k] > 0.0) {
        if (th2 >= run && th2 < run + mx[k]) atomicMin(&s_hit, c0 + k);
        last = c0 + k;
      }
      run += mx[k];
    }
    if (last >= 0) atomicMax(&s_last, last);
    __syncthreads();
    const int col = s_hit != 0x7fffffff ? s_hit : s_last;
    if (col >= 0) pick = d.col0 + col;
  }
  if (tid == 0) {
    a.accepted[b] = acc;
    a.next_token[b] = pick;
    a.status[b] = pick >= 0 ? 0 : TT_REQ_NOT_FINITE;
  }
}

}  // namespace

constexpr size_t kWorkBlockBytes = size_t(kWorkShards) * kWorkStride * sizeof(unsigned long long);

ShardWorkspace shard_layout(void* base, int64_t rows, int S, const int32_t* nch) {
  ShardWorkspace w;
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    char* r = p ? p + off : nullptr;
    off = align256(off + n);
    return r;
  };
  for (int s = 0; s < TT_MAX_SHARDS; ++s)
    w.part[s] = s < S ? reinterpret_cast<Partial*>(take(sizeof(Partial) * size_t(rows) * nch[s]))
                      : nullptr;
  w.excl = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * size_t(S) * rows));
  w.rec = reinterpret_cast<ShardRec*>(take(sizeof(ShardRec) * size_t(S) * rows));
  w.work = reinterpret_cast<unsigned long long*>(take(kWorkBlockBytes * S));
  w.err = reinterpret_cast<int32_t*>(take(2 * sizeof(int32_t)));
  w.bytes = off;
  return w;
}

cudaError_t launch_shard_excl(const ShardArgs& args, cudaStream_t stream) {
  const int64_t n = std::max<int64_t>(args.rows, int64_t(kWorkShards) * kWorkStride * args.S);
  const int blocks = int(std::min<int64_t>((n + 255) / 256, 4096));
  shard_excl_kernel<<<blocks, 256, 0, stream>>>(args, const_cast<int32_t*>(args.err));
  return cudaGetLastError();
}

cudaError_t launch_shard_summary(const ShardArgs& args, cudaStream_t stream, int sm_count) {
  const int64_t warps = int64_t(args.S) * args.rows;
  if (warps == 0) return cudaSuccess;
  const int blocks = int(std::min<int64_t>((warps + 7) / 8, int64_t(sm_count) * 8));
  shard_summary_kernel<<<blocks, 256, 0, stream>>>(args);
  return cudaGetLastError();
}

cudaError_t launch_decide_sharded(const ShardArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  decide_sharded_kernel<<<args.B, kShThreads, 0, stream>>>(args);
  return cudaGetLastError();
}

cudaError_t preload_shard() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, shard_excl_kernel)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, shard_summary_kernel)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, decide_sharded_kernel);
}

}  // namespace tt
