// decide.cu -- per-request decision of one verification step (§4.2, Alg. 2
// accept loop, Alg. 4 residual) and the standalone transfer (Alg. 2
// MapProbabilities, App. A.2).
//
// One CTA per request. From the row-pass partials it rebuilds, in fp64, the
// log2-normaliser of each of the m+1 target rows (adding back the scored
// token's term exactly) and of each mapped draft row, giving p(t_j) and the
// transferred q(t_j). Thread 0 runs the sequential accept loop with Philox
// uniforms. The next token is drawn by a two-level inverse CDF over row a:
// the chunk is found from the partials' masses, then only that chunk of
// kChunk logits is re-read and scanned in column order.
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

constexpr int kWarps = kRowThreads / 32;
constexpr int kRun = kChunk / kRowThreads;  // contiguous columns per thread in the re-read

__device__ __forceinline__ float load_any(const RowSet& R, int dt, int64_t row, int64_t col) {
  const void* p = R.data + row * R.stride_bytes;
  return dt == TT_F32 ? load_logit<TT_F32>(p, col) : load_logit<TT_BF16>(p, col);
}

// exp2 of an fp32 exponent computed as z * scale - M in one rounding.
__device__ __forceinline__ float mass(float z, float scale, float M) {
  return ex2_approx(fmaf(z, scale, -M));
}

// log2-normaliser of a draft row (its partials include every column) and the
// probability of column col under it; computed by one warp.
__device__ __forceinline__ double draft_prob_warp(const DecideArgs& a, int64_t row, int col,
                                                  int lane, bool& finite) {
  float M;
  double S;
  row_norm_warp(a.d.part + row * a.d.nch, a.d.nch, lane, M, S);
  const double x = double(load_any(a.d, a.dt_d, row, col)) * double(a.d.scale);
  const double lse2 = double(M) + log2(S);
  finite = isfinite(lse2);
  return exp2(x - lse2);
}

__device__ __forceinline__ int block_or(int v) { return __syncthreads_or(v); }

// Prefix sums over the block in fp64. The exclusive value of a thread is the
// inclusive value of the one before it, so consecutive runs tile exactly.
__device__ __forceinline__ void block_scan(double v, double* s_warp, double& excl, double& incl,
                                           double& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double n = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += n;
  }
  const double prev = __shfl_up_sync(0xffffffffu, v, 1);
  if (lane == 31) s_warp[warp] = v;
  __syncthreads();
  double before = 0.0, tot = 0.0;
  for (int w = 0; w < kWarps; ++w) {
    if (w < warp) before += s_warp[w];
    tot += s_warp[w];
  }
  __syncthreads();
  incl = before + v;
  excl = lane == 0 ? before : before + prev;
  total = tot;
}

__global__ void __launch_bounds__(kRowThreads) decide_kernel(DecideArgs a) {
  __shared__ double s_p[TT_MAX_M], s_q[TT_MAX_M];
  __shared__ float s_M[TT_MAX_M + 1];   // fp32 reference maximum of each target row
  __shared__ double s_S[TT_MAX_M + 1];  // sum of 2^(s_x - s_M) over the whole row
  __shared__ double s_R[kMaxChunksPerRow];
  __shared__ double s_warp[kWarps];
  __shared__ int s_a, s_chunk, s_pick, s_last;
  __shared__ double s_theta;
  __shared__ float s_dM;
  __shared__ double s_dS;

  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool want_draft = a.full_q || a.q_hat_in == nullptr;
  if (tid == 0) {
    s_dM = 0.f;
    s_dS = 1.0;
  }

  // ------------------------------------------------------------- checks
  int st = a.status_in ? a.status_in[b] : 0;
  int t0 = 0, m = 0, d0 = 0, k = 0;
  if (st == 0) {
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
  }
  if (st == 0) {
    int bad = 0;
    for (int j = tid; j < m; j += kRowThreads) {
      const int col = a.target_cols[t0 + j];
      if (col < 0 || col >= a.t.V) bad = 1;
      if (want_draft) {
        const int i = a.map[t0 + j];
        if (i < 0 || i >= k) bad = 1;
      }
    }
    if (a.q_hat_in == nullptr && a.draft_probs == nullptr)
      for (int i = tid; i < k; i += kRowThreads) {
        const int col = a.draft_cols[d0 + i];
        if (col < 0 || col >= a.d.V) bad = 1;
      }
    if (block_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  }
  if (st != 0) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = st;
    }
    return;
  }

  // ------------------------------------- target rows: normalisers and p(t_j)
  int nonfinite = 0;
  for (int j = warp; j <= m; j += kWarps) {
    const int64_t row = int64_t(t0) + b + j;
    float M;
    double S;
    row_norm_warp(a.t.part + row * a.t.nch, a.t.nch, lane, M, S);
    double lse2, ph = 0.0;
    if (j < m) {  // add back the scored token's term, left out by the row pass
      const double x = double(load_any(a.t, a.dt_t, row, a.target_cols[t0 + j])) *
                       double(a.t.scale);
      const float Mx = fmaxf(M, float(x));  // reference maximum including the token
      S = (M == -INFINITY ? 0.0 : S * exp2(double(M) - double(Mx))) + exp2(x - double(Mx));
      M = Mx;
      lse2 = double(M) + log2(S);
      ph = exp2(x - lse2);
    } else {
      lse2 = double(M) + log2(S);
    }
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
  }

  // ------------------------------------------- transferred draft probability
  for (int j = warp; j < m; j += kWarps) {
    double qh;
    if (a.q_hat_in) {
      qh = double(a.q_hat_in[t0 + j]);
    } else {
      const int64_t row = int64_t(d0) + a.map[t0 + j];
      if (a.draft_probs) {
        qh = double(a.draft_probs[row]);
      } else {
        bool fin;
        qh = draft_prob_warp(a, row, a.draft_cols[row], lane, fin);
        if (!fin) nonfinite = 1;
      }
    }
    if (lane == 0) {
      s_q[j] = qh;
      if (a.q_hat_out) a.q_hat_out[t0 + j] = float(qh);
    }
  }
  if (block_or(nonfinite)) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = TT_REQ_NOT_FINITE;
    }
    return;
  }

  // ------------------------------------------------ accept (sequential scan)
  if (tid == 0) {
    int acc = 0;
    const uint64_t req = a.request_base + uint64_t(b);
    for (int j = 0; j < m; ++j) {
      const double u = philox_uniform(a.seed, uint64_t(j), 0, req);
      const double p = s_p[j], q = s_q[j];
      const double ratio = q > 0.0 ? p / q : (p > 0.0 ? INFINITY : 0.0);
      if (u < fmin(1.0, ratio)) ++acc;
      else break;
    }
    s_a = acc;
  }
  __syncthreads();
  const int acc = s_a;
  const int64_t row = int64_t(t0) + b + acc;
  const int col_t = acc < m ? a.target_cols[t0 + acc] : -1;
  const float Mt = s_M[acc];
  const double St = s_S[acc];
  const float invSt = float(1.0 / St);
  const float scale_t = a.t.scale;
  const char* trow = a.t.data + row * a.t.stride_bytes;
  const int nch = a.t.nch;

  // mode 0: the row's own distribution; 1: one-hot residual; 2: full-q residual
  int mode = acc < m ? (a.full_q ? 2 : 1) : 0;
  const double r_t = acc < m ? fmax(0.0, s_p[acc] - s_q[acc]) : 0.0;
  const char* drow = nullptr;
  if (mode == 2) {
    if (warp == 0) {
      const int64_t rd = int64_t(d0) + a.map[t0 + acc];
      float M;
      double S;
      row_norm_warp(a.d.part + rd * a.d.nch, a.d.nch, lane, M, S);
      if (lane == 0) {
        s_dM = M;
        s_dS = S;
      }
    }
    drow = a.d.data + (int64_t(d0) + a.map[t0 + acc]) * a.d.stride_bytes;
  }
  __syncthreads();
  const float Md = s_dM;
  const float invSd = mode == 2 ? float(1.0 / s_dS) : 0.f;
  const float scale_d = a.d.scale;

  // residual mass of column x of row `row` in the current mode (fp32)
  auto r_of = [&](int x, int md) -> float {
    const float z = a.dt_t == TT_F32 ? __ldg(reinterpret_cast<const float*>(trow) + x)
                                     : bf16_to_f32(__ldg(reinterpret_cast<const unsigned short*>(trow) + x));
    const float p = mass(z, scale_t, Mt) * invSt;
    if (md == 1) return x == col_t ? float(r_t) : p;
    if (md == 2) {
      const float zd = a.dt_d == TT_F32 ? __ldg(reinterpret_cast<const float*>(drow) + x)
                                        : bf16_to_f32(__ldg(reinterpret_cast<const unsigned short*>(drow) + x));
      const float q = mass(zd, scale_d, Md) * invSd;
      return fmaxf(0.f, p - q);
    }
    return p;
  };

  // ----------------------------------------- coarse level: mass per chunk
  for (int pass = 0; pass < 2; ++pass) {
    if (mode == 2) {
      for (int c = 0; c < nch; ++c) {
        const int x0 = c * kChunk + tid * kRun, x1 = min(x0 + kRun, a.t.V);
        float part = 0.f;
        for (int x = x0; x < x1; ++x) part += r_of(x, 2);
        double e, i, tot;
        block_scan(double(part), s_warp, e, i, tot);
        if (tid == 0) s_R[c] = tot;
      }
    } else {
      for (int c = tid; c < nch; c += kRowThreads) {
        const Partial P = a.t.part[row * nch + c];
        double R = P.m == -INFINITY ? 0.0 : double(P.s) * exp2(double(P.m) - double(Mt)) / St;
        if (col_t >= 0 && col_t / kChunk == c) R += mode == 1 ? r_t : s_p[acc];
        s_R[c] = R;
      }
    }
    __syncthreads();
    if (tid == 0) {
      double Z = 0.0;
      for (int c = 0; c < nch; ++c) Z += s_R[c];
      s_theta = Z;
    }
    __syncthreads();
    if (s_theta > 0.0 || mode == 0) break;
    __syncthreads();
    mode = 0;  // degenerate residual (rounding): fall back to the row itself
  }

  if (tid == 0) {
    const double Z = s_theta;
    const double u = philox_uniform(a.seed, uint64_t(acc), 1, a.request_base + uint64_t(b));
    const double theta = u * Z;
    double cum = 0.0;
    int pick = -1, last = -1;
    double base_pick = 0.0, base_last = 0.0;
    for (int c = 0; c < nch; ++c) {
      if (s_R[c] > 0.0) {
        last = c;
        base_last = cum;
      }
      if (pick < 0 && cum + s_R[c] > theta) {
        pick = c;
        base_pick = cum;
      }
      cum += s_R[c];
    }
    if (pick < 0) {  // theta at the very top (rounding): the last chunk with mass
      pick = last < 0 ? 0 : last;
      base_pick = base_last;
      s_theta = INFINITY;
    } else {
      s_theta = theta - base_pick;
    }
    s_chunk = pick;
    s_pick = -1;
    s_last = -1;
  }
  __syncthreads();

  // ------------------------------------------- fine level: one chunk re-read
  const double theta = s_theta;
  const int x0 = s_chunk * kChunk + tid * kRun, x1 = min(x0 + kRun, a.t.V);
  float run = 0.f;
  int last_pos = -1;
  for (int x = x0; x < x1; ++x) {
    const float r = r_of(x, mode);
    run += r;
    if (r > 0.f) last_pos = x;
  }
  double excl, incl, tot;
  block_scan(double(run), s_warp, excl, incl, tot);
  if (excl <= theta && theta < incl) {  // the running mass crosses theta in this run
    double c = excl;
    int pick = last_pos;
    for (int x = x0; x < x1; ++x) {
      c += double(r_of(x, mode));
      if (c > theta) {
        pick = x;
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
__global__ void __launch_bounds__(kRowThreads) transfer_kernel(DecideArgs a) {
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int st = 0;
  if (!csr_ok(a.target_off, b, a.n_target) || !csr_ok(a.draft_off, b, a.n_draft)) {
    if (tid == 0) a.status[b] = TT_REQ_BAD_OFFSETS;
    return;
  }
  const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
  const int d0 = a.draft_off[b], k = a.draft_off[b + 1] - d0;
  if (m == 0 || k == 0) st = TT_REQ_EMPTY;
  int bad = 0;
  if (st == 0) {
    for (int j = tid; j < m; j += kRowThreads) {
      const int i = a.map[t0 + j];
      if (i < 0 || i >= k) bad = 1;
    }
    if (a.draft_probs == nullptr)
      for (int i = tid; i < k; i += kRowThreads) {
        const int col = a.draft_cols[d0 + i];
        if (col < 0 || col >= a.d.V) bad = 1;
      }
  }
  if (block_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st != 0) {
    for (int j = tid; j < m; j += kRowThreads) a.q_hat_out[t0 + j] = 0.f;
    if (tid == 0) a.status[b] = st;
    return;
  }
  int nonfinite = 0;
  for (int j = warp; j < m; j += kWarps) {
    const int64_t row = int64_t(d0) + a.map[t0 + j];
    double qh;
    if (a.draft_probs) {
      qh = double(a.draft_probs[row]);
    } else {
      bool fin;
      qh = draft_prob_warp(a, row, a.draft_cols[row], lane, fin);
      if (!fin) nonfinite = 1;
    }
    if (lane == 0) a.q_hat_out[t0 + j] = float(qh);
  }
  const int nf = block_or(nonfinite);
  if (tid == 0) a.status[b] = nf ? TT_REQ_NOT_FINITE : 0;
}

// Needed-draft-row flags from a map, and the scored column of each target row.
__global__ void prep_kernel(PrepArgs a) {
  const int b = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (b >= a.B) return;
  if (a.excl && csr_ok(a.target_off, b, a.n_target)) {
    const int t0 = a.target_off[b], m = a.target_off[b + 1] - t0;
    for (int j = lane; j <= m; j += 32) {
      int col = -1;
      if (j < m) {
        const int c = a.target_cols[t0 + j];
        col = (c >= 0 && c < a.V_t) ? c : -1;
      }
      a.excl[t0 + b + j] = col;
    }
  }
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

}  // namespace

cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  if (args.mode_transfer_only)
    transfer_kernel<<<args.B, kRowThreads, 0, stream>>>(args);
  else
    decide_kernel<<<args.B, kRowThreads, 0, stream>>>(args);
  return cudaGetLastError();
}

cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  constexpr int kWarpsPerBlock = 4;
  prep_kernel<<<(args.B + kWarpsPerBlock - 1) / kWarpsPerBlock, 32 * kWarpsPerBlock, 0, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace tt
