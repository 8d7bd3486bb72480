// decide.cu -- per-request decision of one verification step (§4.2, Alg. 2
// accept loop, Alg. 4 residual) and the standalone transfer (Alg. 2
// MapProbabilities, App. A.2).
//
// One CTA per request. From the row-pass partials it rebuilds, in fp64, the
// log2-normaliser of each of the m+1 target rows (adding back the scored
// token's term exactly) and of each mapped draft row, giving p(t_j) and the
// transferred q(t_j). The accept uniforms are drawn in parallel, one thread per
// position; the first rejection is the smallest failing position. The next
// token is drawn by a two-level inverse CDF over row a: the chunk comes from
// the partials' masses, then only that chunk of kChunk logits is re-read.
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

constexpr int kDecThreads = 512;
constexpr int kWarps = kDecThreads / 32;
constexpr int kPer = kChunk / kDecThreads;  // columns per thread in the re-read
static_assert(kDecThreads >= TT_MAX_M, "one thread per target position");

__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

__device__ __forceinline__ float load_dt(const char* row, int dt, int64_t col) {
  return dt == TT_F32 ? load_logit<TT_F32>(row, col) : load_logit<TT_BF16>(row, col);
}

// A logit of row `row` of a family, read only after a bounds check; a failed
// check is recorded and reads as -inf.
__device__ __forceinline__ float load_checked(const DecideArgs& a, const RowSet& R, int dt,
                                              int64_t row, int64_t col) {
  if (row < 0 || row >= R.n_rows || col < 0 || col >= R.V) {
    report_error(a.err, a.epoch, TT_REQ_INTERNAL);
    return -INFINITY;
  }
  return load_dt(R.data + row * R.stride_bytes, dt, col);
}

// Prefix sums over the block in fp64; the exclusive value of a thread is the
// inclusive value of the one before it, so consecutive ranges tile exactly.
__device__ __forceinline__ void block_scan(double v, double* s_warp, double& excl, double& incl) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  const double prev = __shfl_up_sync(0xffffffffu, v, 1);
  if (lane == 31) s_warp[warp] = v;
  __syncthreads();
  double before = 0.0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) before += w < warp ? s_warp[w] : 0.0;
  __syncthreads();
  incl = before + v;
  excl = lane == 0 ? before : before + prev;
}

// Inclusive prefix sum over a warp in fp64.
__device__ __forceinline__ double warp_scan_d(double v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  return v;
}

__device__ __forceinline__ void fail(const DecideArgs& a, int b, int st) {
  if (threadIdx.x == 0) {
    a.accepted[b] = 0;
    a.next_token[b] = -1;
    a.status[b] = st;
  }
}

__global__ void __launch_bounds__(kDecThreads) decide_kernel(DecideArgs a) {
  __shared__ double s_p[TT_MAX_M], s_q[TT_MAX_M];
  __shared__ int s_col[TT_MAX_M], s_map[TT_MAX_M];
  __shared__ float s_M[TT_MAX_M + 1];   // fp32 reference maximum of each target row
  __shared__ double s_S[TT_MAX_M + 1];  // sum over the row of 2^(s_x - s_M)
  __shared__ double s_R[kMaxChunksPerRow];
  __shared__ double s_warp[kWarps];
  __shared__ int s_a, s_chunk, s_pick, s_last;
  __shared__ double s_theta;
  __shared__ float s_dM;
  __shared__ double s_dS;

  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool want_draft = a.full_q || a.q_hat_in == nullptr;
  const bool q_from_logits = a.q_hat_in == nullptr && a.draft_probs == nullptr;

  // ------------------------------------------ checks on the caller's inputs
  int st = 0, t0 = 0, m = 0, d0 = 0, k = 0;
  if (!csr_ok(a.target_off, b, a.n_target) ||
      (want_draft && !csr_ok(a.draft_off, b, a.n_draft))) {
    st = TT_REQ_BAD_OFFSETS;
  } else {
    t0 = a.target_off[b];
    m = a.target_off[b + 1] - t0;
    if (want_draft) {
      d0 = a.draft_off[b];
      k = a.draft_off[b + 1] - d0;
    }
    if (m == 0 || (want_draft && k == 0)) st |= TT_REQ_EMPTY;
    if (m > a.max_m || m > TT_MAX_M) st |= TT_REQ_TOO_LONG;
  }
  if (tid == 0) {
    s_a = m;
    s_pick = -1;
    s_last = -1;
    s_dM = 0.f;
    s_dS = 1.0;
  }
  int bad = 0;
  if (st == 0) {
    for (int j = tid; j < m; j += kDecThreads) {
      const int col = a.target_cols[t0 + j];
      s_col[j] = col;
      if (col < 0 || col >= a.t.V) bad = 1;
    }
    if (q_from_logits)
      for (int i = tid; i < k; i += kDecThreads) {
        const int col = a.draft_cols[d0 + i];
        if (col < 0 || col >= a.d.V) bad = 1;
      }
  }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;

  // ------------------------------ results of the kernels before this one
  grid_dependency_wait();
  if (a.status_in) {
    const int s_in = a.status_in[b];
    if (s_in != 0) st = s_in;  // the alignment's verdict comes first
  }
  if (a.err && a.err[0] == a.epoch) st = a.err[1];  // the row pass failed
  bad = 0;
  if (st == 0 && want_draft)
    for (int j = tid; j < m; j += kDecThreads) {
      const int i = a.map[t0 + j];
      s_map[j] = i;
      if (i < 0 || i >= k) bad = 1;
    }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st != 0) {
    fail(a, b, st);
    return;
  }

  // ------------- normalisers: target rows 0..m, then each run's draft row
  int nonfinite = 0;
  const int n_tasks = m + 1 + (q_from_logits ? m : 0);
  for (int task = warp; task < n_tasks; task += kWarps) {
    if (task <= m) {
      const int j = task;
      const int64_t row = int64_t(t0) + b + j;
      const float zt = j < m ? load_checked(a, a.t, a.dt_t, row, s_col[j]) : 0.f;
      float M;
      double S;
      row_norm_warp(a.t.part + row * a.t.nch, a.t.nch, lane, M, S);
      double lse2, ph = 0.0;
      if (j < m) {  // add back the scored token's term, left out by the row pass
        const double x = double(zt) * double(a.t.scale);
        const float Mx = fmaxf(M, float(x));
        S = (M == -INFINITY ? 0.0 : S * exp2_split(double(M) - double(Mx))) +
            exp2_split(x - double(Mx));
        M = Mx;
        ph = exp2_split(x - double(M)) * double(__frcp_rn(float(S)));
      }
      lse2 = double(M) + log2_split(S);
      if (!isfinite(lse2)) nonfinite = 1;
      if (lane == 0) {
        s_M[j] = M;
        s_S[j] = S;
        if (j < m) {
          s_p[j] = ph;
          if (a.p_hat) a.p_hat[t0 + j] = float(ph);
        }
        if (a.lse) a.lse[row] = float(lse2 * 0.69314718055994530942);
      }
    } else {
      const int j = task - (m + 1);
      if (j > 0 && s_map[j] == s_map[j - 1]) continue;  // copy rule: same draft row
      const int64_t row = int64_t(d0) + s_map[j];
      const float zd = load_checked(a, a.d, a.dt_d, row, a.draft_cols[row]);
      float M;
      double S;
      row_norm_warp(a.d.part + row * a.d.nch, a.d.nch, lane, M, S);
      if (!(S > 0.0) || !isfinite(S) || M == -INFINITY) nonfinite = 1;
      if (lane == 0)
        s_q[j] = exp2_split(double(zd) * double(a.d.scale) - double(M)) *
                 double(__frcp_rn(float(S)));
    }
  }
  if (__syncthreads_or(nonfinite)) {
    fail(a, b, TT_REQ_NOT_FINITE);
    return;
  }
  for (int j = tid; j < m; j += kDecThreads) {
    double qh;
    if (a.q_hat_in) {
      qh = double(a.q_hat_in[t0 + j]);
    } else if (a.draft_probs) {
      qh = double(a.draft_probs[int64_t(d0) + s_map[j]]);
    } else {
      int f = j;  // first position of this run of equal map entries (computed above)
      while (f > 0 && s_map[f - 1] == s_map[j]) --f;
      qh = s_q[f];
    }
    if (a.q_hat_out) a.q_hat_out[t0 + j] = float(qh);
    if (!q_from_logits) s_q[j] = qh;
  }
  __syncthreads();
  if (q_from_logits) {  // fill the runs (their first entries are final)
    for (int j = tid; j < m; j += kDecThreads) {
      int f = j;
      while (f > 0 && s_map[f - 1] == s_map[j]) --f;
      if (f != j) s_q[j] = s_q[f];
    }
    __syncthreads();
  }

  // ------------------------- accept: u_j < min(1, p/q), first failure stops
  const uint64_t req = a.request_base + uint64_t(b);
  if (tid < m) {  // for u < 1, u < min(1, p/q) holds exactly when u q < p
    const double u = philox_uniform(a.seed, uint64_t(tid), 0, req);
    if (!(u * s_q[tid] < s_p[tid])) atomicMin(&s_a, tid);
  }
  __syncthreads();
  const int acc = s_a;
  const int64_t row = int64_t(t0) + b + acc;
  const int col_t = acc < m ? s_col[acc] : -1;
  const float Mt = s_M[acc];
  const double St = s_S[acc];
  const float invSt = __frcp_rn(float(St));
  const float scale_t = a.t.scale;
  const char* trow = a.t.data + row * a.t.stride_bytes;
  const int nch = a.t.nch;
  const int V = a.t.V;
  const double r_t = acc < m ? fmax(0.0, s_p[acc] - s_q[acc]) : 0.0;

  // mode 0: the row's own distribution; 1: one-hot residual; 2: full-q residual
  int mode = acc < m ? (a.full_q ? 2 : 1) : 0;
  const char* drow = nullptr;
  if (mode == 2) {
    const int64_t rd = int64_t(d0) + s_map[acc];
    drow = a.d.data + rd * a.d.stride_bytes;
    if (warp == 0) {
      float M;
      double S;
      row_norm_warp(a.d.part + rd * a.d.nch, a.d.nch, lane, M, S);
      if (lane == 0) {
        s_dM = M;
        s_dS = S;
      }
    }
    __syncthreads();
  }
  const float Md = s_dM;
  const float invSd = __frcp_rn(float(s_dS));
  const float scale_d = a.d.scale;
  // residual mass of column x (logit z) of row a in mode md, fp32
  auto r_of = [&](int x, float z, int md) -> float {
    const float p = ex2_approx(fmaf(z, scale_t, -Mt)) * invSt;
    if (md == 1) return x == col_t ? float(r_t) : p;
    if (md == 2) {
      const float q = ex2_approx(fmaf(load_dt(drow, a.dt_d, x), scale_d, -Md)) * invSd;
      return fmaxf(0.f, p - q);
    }
    return p;
  };
  const double u2 = philox_uniform(a.seed, uint64_t(acc), 1, req);

  // ----------------------------------------- coarse level: mass per chunk
  for (int pass = 0; pass < 2; ++pass) {
    if (mode == 2) {  // elementwise residual, one warp per chunk
      for (int c = warp; c < nch; c += kWarps) {
        float part = 0.f;
        const int hi = min(V, (c + 1) * kChunk);
        for (int x = c * kChunk + lane; x < hi; x += 32) part += r_of(x, load_dt(trow, a.dt_t, x), 2);
        const double tot = warp_sum_d(double(part));
        if (lane == 0) s_R[c] = tot;
      }
    } else {
      for (int c = tid; c < nch; c += kDecThreads) {
        const Partial P = a.t.part[row * nch + c];
        double R = P.m == -INFINITY ? 0.0 : double(P.s * ex2_approx(P.m - Mt) * invSt);
        if (col_t >= 0 && col_t / kChunk == c) R += mode == 1 ? r_t : s_p[acc];
        s_R[c] = R;
      }
    }
    __syncthreads();
    if (warp == 0) {
      // lane-contiguous ranges of chunks, scanned in column order
      const int per = (nch + 31) / 32;
      const int lo = min(nch, lane * per), hi = min(nch, lo + per);
      double loc = 0.0;
      int last = -1;
      for (int c = lo; c < hi; ++c) {
        loc += s_R[c];
        if (s_R[c] > 0.0) last = c;
      }
      const double incl = warp_scan_d(loc, lane);
      const double prev = __shfl_up_sync(0xffffffffu, incl, 1);
      const double excl = lane == 0 ? 0.0 : prev;
      const double Z = __shfl_sync(0xffffffffu, incl, 31);
      int last_all = last;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) last_all = max(last_all, __shfl_xor_sync(0xffffffffu, last_all, o));
      if (!(Z > 0.0) && mode != 0) {
        if (lane == 0) s_chunk = -2;  // degenerate residual
      } else {
        const double theta = u2 * Z;
        int found = -1;
        double rel = INFINITY;
        if (excl <= theta && theta < incl) {
          double cum = excl;
          for (int c = lo; c < hi; ++c) {
            if (theta < cum + s_R[c]) {
              found = c;
              rel = theta - cum;
              break;
            }
            cum += s_R[c];
          }
          if (found < 0) found = last;  // rounding inside the range: its last chunk with mass
        }
        const unsigned hit = __ballot_sync(0xffffffffu, found >= 0);
        if (hit) {
          const int src = __ffs(hit) - 1;
          const int fc = __shfl_sync(0xffffffffu, found, src);
          const double fr = __shfl_sync(0xffffffffu, rel, src);
          if (lane == 0) {
            s_chunk = fc;
            s_theta = fr;
          }
        } else if (lane == 0) {  // theta at the very top: the last chunk with mass
          s_chunk = last_all < 0 ? 0 : last_all;
          s_theta = INFINITY;
        }
      }
    }
    __syncthreads();
    if (s_chunk != -2) break;
    mode = 0;  // fall back to the row itself
    __syncthreads();
  }
  const int chunk = s_chunk;
  const double theta = s_theta;

  // ------------------------------------------ fine level: one chunk re-read
  const int x0 = chunk * kChunk + tid * kPer;
  float r[kPer];
  float run = 0.f;
  int last_pos = -1;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int x = x0 + q;
    float v = 0.f;
    if (x < V) {
      v = r_of(x, load_dt(trow, a.dt_t, x), mode);
      if (v > 0.f) last_pos = x;
    }
    r[q] = v;
    run += v;
  }
  double excl, incl;
  block_scan(double(run), s_warp, excl, incl);
  if (excl <= theta && theta < incl) {
    double c = excl;
    int pick = last_pos;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      c += double(r[q]);
      if (c > theta && r[q] > 0.f) {
        pick = x0 + q;
        break;
      }
    }
    s_pick = pick;
  }
  if (last_pos >= 0) atomicMax(&s_last, last_pos);
  __syncthreads();
  if (tid == 0) {
    a.accepted[b] = acc;
    a.next_token[b] = s_pick >= 0 ? s_pick : s_last;
    a.status[b] = 0;
  }
}

// Standalone transfer: q_hat[j] for every target position of request b.
__global__ void __launch_bounds__(kDecThreads) transfer_kernel(DecideArgs a) {
  __shared__ int s_map[TT_MAX_M];
  __shared__ double s_q[TT_MAX_M];
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int st = 0, t0 = 0, m = 0, d0 = 0, k = 0;
  if (!csr_ok(a.target_off, b, a.n_target) || !csr_ok(a.draft_off, b, a.n_draft)) {
    st = TT_REQ_BAD_OFFSETS;
  } else {
    t0 = a.target_off[b];
    m = a.target_off[b + 1] - t0;
    d0 = a.draft_off[b];
    k = a.draft_off[b + 1] - d0;
    if (m == 0 || k == 0) st = TT_REQ_EMPTY;
    if (m > TT_MAX_M) st |= TT_REQ_TOO_LONG;
  }
  int bad = 0;
  if (st == 0 && a.draft_probs == nullptr)
    for (int i = tid; i < k; i += kDecThreads) {
      const int col = a.draft_cols[d0 + i];
      if (col < 0 || col >= a.d.V) bad = 1;
    }
  grid_dependency_wait();
  if (st == 0)
    for (int j = tid; j < m; j += kDecThreads) {
      const int i = a.map[t0 + j];
      s_map[j] = i;
      if (i < 0 || i >= k) bad = 1;
    }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st == 0 && a.err && a.err[0] == a.epoch) st = a.err[1];
  if (st != 0) {
    if (!(st & (TT_REQ_BAD_OFFSETS | TT_REQ_TOO_LONG)))
      for (int j = tid; j < m; j += kDecThreads) a.q_hat_out[t0 + j] = 0.f;
    if (tid == 0) a.status[b] = st;
    return;
  }
  int nonfinite = 0;
  for (int j = warp; j < m; j += kWarps) {
    if (j > 0 && s_map[j] == s_map[j - 1]) continue;
    const int64_t row = int64_t(d0) + s_map[j];
    double qh;
    if (a.draft_probs) {
      qh = double(a.draft_probs[row]);
    } else {
      const float zd = load_checked(a, a.d, a.dt_d, row, a.draft_cols[row]);
      float M;
      double S;
      row_norm_warp(a.d.part + row * a.d.nch, a.d.nch, lane, M, S);
      if (!(S > 0.0) || !isfinite(S) || M == -INFINITY) nonfinite = 1;
      qh = exp2_split(double(zd) * double(a.d.scale) - double(M)) * double(__frcp_rn(float(S)));
    }
    if (lane == 0) s_q[j] = qh;
  }
  const int nf = __syncthreads_or(nonfinite);
  for (int j = tid; j < m; j += kDecThreads) {
    int f = j;
    while (f > 0 && s_map[f - 1] == s_map[j]) --f;
    a.q_hat_out[t0 + j] = float(s_q[f]);
  }
  if (tid == 0) a.status[b] = nf ? TT_REQ_NOT_FINITE : 0;
}

// Needed-draft-row flags from an alignment map.
__global__ void prep_kernel(PrepArgs a) {
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (b >= a.B) return;
  if (a.need && csr_ok(a.draft_off, b, a.n_draft) && csr_ok(a.target_off, b, a.n_target)) {
    const int d0 = a.draft_off[b], k = a.draft_off[b + 1] - d0;
    const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
    for (int i = lane; i < k; i += 32) a.need[d0 + i] = 0;
    __syncwarp();
    for (int j = lane; j < m; j += 32) {
      const int i = a.map[t0 + j];
      if (i >= 0 && i < k) a.need[d0 + i] = 1;
    }
  }
}

template <typename K>
cudaError_t launch_pdl(K kernel, const DecideArgs& args, cudaStream_t stream, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(args.B));
  cfg.blockDim = dim3(kDecThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args);
}

}  // namespace

cudaError_t preload_decide() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, decide_kernel)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, transfer_kernel)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, prep_kernel);
}

cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (args.B == 0) return cudaSuccess;
  if (args.mode_transfer_only) return launch_pdl(transfer_kernel, args, stream, pdl);
  return launch_pdl(decide_kernel, args, stream, pdl);
}

cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  constexpr int kWarpsPerBlock = 4;
  prep_kernel<<<(args.B + kWarpsPerBlock - 1) / kWarpsPerBlock, 32 * kWarpsPerBlock, 0, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace tt
