// decide.cu -- per-request decision of one verification step (§4.2, Alg. 2
// accept loop, Alg. 4 residual) and the standalone transfer (Alg. 2
// MapProbabilities, App. A.2).
//
// One CTA per request. From the row-pass partials it rebuilds the
// log2-normaliser of each of the m+1 target rows (adding back the scored
// token's term) and of each mapped draft row, giving p(t_j) and the
// transferred q(t_j); fp32 with compensated sums and exactly split exponents,
// since fp64 transcendentals are slow on this part. The accept uniforms are drawn in parallel, one thread per
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

// ------------------------------------------------------------------------
// Arithmetic of the decision kernel. Row normalisers are fp32 with compensated
// (TwoSum) reductions and exactly split exponents; the prefix scans that pick
// the next token run in fp64.

struct F2 {  // unevaluated sum hi + lo
  float hi, lo;
};

__device__ __forceinline__ F2 two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  return {s, __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb))};
}

__device__ __forceinline__ F2 f2_add(F2 a, F2 b) {
  const F2 s = two_sum(a.hi, b.hi);
  const float lo = __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo));
  const float hi = __fadd_rn(s.hi, lo);
  return {hi, __fsub_rn(lo, __fsub_rn(hi, s.hi))};
}

// Compensated sum over the warp; every lane gets lane 0's result.
__device__ __forceinline__ float warp_sum_comp(F2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const F2 w = {__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)};
    v = f2_add(v, w);
  }
  return __shfl_sync(0xffffffffu, __fadd_rn(v.hi, v.lo), 0);
}

// 2^(z * scale - M) with the exponent split exactly into n + f, |f| <= 1/2:
// z * scale = xh + xl and xh - M = dh + dl are error-free transformations, so
// only 2^f (from the SFU, relative error about 2^-22) is approximate.
__device__ __forceinline__ float exp2_scaled(float z, float scale, float M) {
  const float xh = __fmul_rn(z, scale);
  const float xl = fmaf(z, scale, -xh);
  const F2 d = two_sum(xh, -M);
  const float n = rintf(d.hi);
  const float f = __fadd_rn(__fsub_rn(d.hi, n), __fadd_rn(d.lo, xl));
  if (!(n > -126.f)) return 0.f;
  return ex2_approx(f) * __int_as_float((int(n) + 127) << 23);
}

// Max and sum of 2^(m_c - max) * s_c of one row's partials (one warp; all
// lanes get the same values). Rows of up to 128 chunks use the cached loads.
__device__ __forceinline__ void row_stats(const Partial* part, int nch, const Partial (&cache)[4],
                                          int lane, float& mx, float& S) {
  float m = -INFINITY;
  F2 acc = {0.f, 0.f};
  if (nch <= 128) {
#pragma unroll
    for (int i = 0; i < 4; ++i) m = fmaxf(m, cache[i].m);
    m = warp_max_f(m);
    if (m != -INFINITY) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (cache[i].m != -INFINITY) acc = f2_add(acc, F2{cache[i].s * ex2_approx(cache[i].m - m), 0.f});
    }
  } else {
    for (int c = lane; c < nch; c += 32) m = fmaxf(m, part[c].m);
    m = warp_max_f(m);
    if (m != -INFINITY)
      for (int c = lane; c < nch; c += 32) {
        const Partial q = part[c];
        if (q.m != -INFINITY) acc = f2_add(acc, F2{q.s * ex2_approx(q.m - m), 0.f});
      }
  }
  mx = m;
  S = warp_sum_comp(acc);
}

__device__ __forceinline__ void load_cache(const Partial* part, int nch, int lane, bool valid,
                                           Partial (&cache)[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int c = lane + 32 * i;
    cache[i] = (valid && nch <= 128 && c < nch) ? part[c] : Partial{-INFINITY, 0.f};
  }
}

struct RowResult {
  float M, S;  // reference maximum and sum of 2^(s - M) over the whole row
};

// Adds the scored token's term (left out by the row pass) to a target row.
__device__ __forceinline__ RowResult with_token(float mx, float S, float zt, float scale) {
  const float xh = __fmul_rn(zt, scale);
  const float Mx = fmaxf(mx, xh);
  const float rest = mx == -INFINITY ? 0.f : S * ex2_approx(mx - Mx);
  return {Mx, rest + exp2_scaled(zt, scale, Mx)};
}

// One CTA (16 warps) per request: the warps share the row normalisers, the
// accept draws run one thread per position, warp 0 picks the chunk and the
// whole CTA re-reads it (4 columns per thread).
__global__ void __launch_bounds__(kDecThreads) decide_kernel(DecideArgs a) {
  __shared__ float s_p[TT_MAX_M], s_q[TT_MAX_M];
  __shared__ int s_col[TT_MAX_M], s_map[TT_MAX_M];
  __shared__ float s_M[TT_MAX_M + 1], s_S[TT_MAX_M + 1];
  __shared__ double s_R[kMaxChunksPerRow];
  __shared__ double s_wtot[kWarps], s_wpre[kWarps];
  __shared__ int s_a, s_chunk, s_pick, s_last;
  __shared__ double s_theta;
  __shared__ float s_dM, s_dS;

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
    s_dS = 1.f;
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
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = st;
    }
    return;
  }

  // ------ row normalisers, one warp per row: target rows 0..m, then the
  // first row of each run of equal map entries (the copy rule reuses it)
  int nonfinite = 0;
  const int n_tasks = m + 1 + (q_from_logits ? m : 0);
  for (int task = warp; task < n_tasks; task += kWarps) {
    const bool tgt = task <= m;
    const int j = tgt ? task : task - (m + 1);
    if (!tgt && j > 0 && s_map[j] == s_map[j - 1]) continue;
    const int64_t row = tgt ? int64_t(t0) + b + j : int64_t(d0) + s_map[j];
    const RowSet& R = tgt ? a.t : a.d;
    const int dt = tgt ? a.dt_t : a.dt_d;
    const Partial* part = R.part + row * R.nch;
    // issue the loads first: the scored token's logit and the row's partials
    float z = 0.f;
    if (!tgt) z = load_checked(a, R, dt, row, a.draft_cols[row]);
    else if (j < m) z = load_checked(a, R, dt, row, s_col[j]);
    Partial cache[4];
    load_cache(part, R.nch, lane, true, cache);
    float mx, S;
    row_stats(part, R.nch, cache, lane, mx, S);
    if (tgt) {
      float M = mx, Stot = S, ph = 0.f;
      if (j < m) {  // add back the scored token's term, left out by the row pass
        const RowResult rr = with_token(mx, S, z, R.scale);
        M = rr.M;
        Stot = rr.S;
        ph = exp2_scaled(z, R.scale, M) * __frcp_rn(Stot);
      }
      if (!(Stot > 0.f) || !isfinite(Stot) || isnan(M)) nonfinite = 1;
      if (lane == 0) {
        s_M[j] = M;
        s_S[j] = Stot;
        if (j < m) {
          s_p[j] = ph;
          if (a.p_hat) a.p_hat[t0 + j] = ph;
        }
        if (a.lse) a.lse[row] = (M + lg2_approx(Stot)) * 0.6931471805599453f;
      }
    } else {
      if (!(S > 0.f) || !isfinite(S) || mx == -INFINITY) nonfinite = 1;
      if (lane == 0) s_q[j] = exp2_scaled(z, R.scale, mx) * __frcp_rn(S);
    }
  }
  if (__syncthreads_or(nonfinite)) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = TT_REQ_NOT_FINITE;
    }
    return;
  }
  for (int j = tid; j < m; j += kDecThreads) {
    float qh;
    if (a.q_hat_in) {
      qh = a.q_hat_in[t0 + j];
    } else if (a.draft_probs) {
      qh = a.draft_probs[int64_t(d0) + s_map[j]];
    } else {
      int f = j;  // first position of this run of equal map entries
      while (f > 0 && s_map[f - 1] == s_map[j]) --f;
      qh = s_q[f];
    }
    if (a.q_hat_out) a.q_hat_out[t0 + j] = qh;
    if (!q_from_logits) s_q[j] = qh;
  }
  __syncthreads();
  if (q_from_logits) {  // copies of a run take the value of its first entry
    for (int j = tid; j < m; j += kDecThreads) {
      int f = j;
      while (f > 0 && s_map[f - 1] == s_map[j]) --f;
      if (f != j) s_q[j] = s_q[f];
    }
    __syncthreads();
  }

  // --------------------------- accept while u_j q_j < p_j (u < 1 exactly)
  const uint64_t req = a.request_base + uint64_t(b);
  if (tid < m) {
    const float u = float(philox_uniform(a.seed, uint64_t(tid), 0, req));
    if (!(u * s_q[tid] < s_p[tid])) atomicMin(&s_a, tid);
  }
  __syncthreads();
  const int acc = s_a;
  const int64_t row = int64_t(t0) + b + acc;
  const int nch = a.t.nch;
  const int V = a.t.V;
  const int col_t = acc < m ? s_col[acc] : -1;
  const float Mt = s_M[acc];
  const float invSt = __frcp_rn(s_S[acc]);
  const float scale_t = a.t.scale;
  const char* trow = a.t.data + row * a.t.stride_bytes;
  const float p_a = acc < m ? s_p[acc] : 0.f;
  const float r_t = acc < m ? fmaxf(0.f, p_a - s_q[acc]) : 0.f;
  int mode = acc < m ? (a.full_q ? 2 : 1) : 0;  // 0 the row itself, 1 one-hot, 2 full-q residual
  const char* drow = nullptr;
  if (mode == 2) {
    const int64_t rd = int64_t(d0) + s_map[acc];
    drow = a.d.data + rd * a.d.stride_bytes;
    if (warp == 0) {
      Partial c4[4];
      load_cache(a.d.part + rd * a.d.nch, a.d.nch, lane, true, c4);
      float Md, Sd;
      row_stats(a.d.part + rd * a.d.nch, a.d.nch, c4, lane, Md, Sd);
      if (lane == 0) {
        s_dM = Md;
        s_dS = Sd;
      }
    }
    __syncthreads();
  }
  const float Md = s_dM;
  const float invSd = __frcp_rn(s_dS);
  auto r_of = [&](int x, float z, int md) -> float {
    const float p = ex2_approx(fmaf(z, scale_t, -Mt)) * invSt;
    if (md == 1) return x == col_t ? r_t : p;
    if (md == 2) {
      const float q = ex2_approx(fmaf(load_dt(drow, a.dt_d, x), a.d.scale, -Md)) * invSd;
      return fmaxf(0.f, p - q);
    }
    return p;
  };
  const double u2 = philox_uniform(a.seed, uint64_t(acc), 1, req);

  // ------------------------------- coarse level: the chunk holding u' * Z
  for (int pass = 0; pass < 2; ++pass) {
    if (mode == 2) {  // elementwise residual masses, one warp per chunk
      for (int c = warp; c < nch; c += kWarps) {
        F2 part = {0.f, 0.f};
        const int hi_c = min(V, (c + 1) * kChunk);
        for (int x = c * kChunk + lane; x < hi_c; x += 32)
          part = f2_add(part, F2{r_of(x, load_dt(trow, a.dt_t, x), 2), 0.f});
        const float Rc = warp_sum_comp(part);
        if (lane == 0) s_R[c] = double(Rc);
      }
    } else {
      for (int c = tid; c < nch; c += kDecThreads) {
        const Partial P = a.t.part[row * nch + c];
        double R = P.m == -INFINITY ? 0.0 : double(P.s * ex2_approx(P.m - Mt) * invSt);
        if (col_t >= 0 && col_t / kChunk == c) R += mode == 1 ? r_t : p_a;
        s_R[c] = R;
      }
    }
    __syncthreads();
    if (warp == 0) {  // lane-contiguous ranges of chunks, scanned in column order
      const int per = (nch + 31) / 32;
      const int lo = min(nch, lane * per), hi = min(nch, lo + per);
      double loc = 0.0;
      int last = -1;
      for (int c = lo; c < hi; ++c) {
        loc += s_R[c];
        if (s_R[c] > 0.0) last = c;
      }
      double incl = loc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const double n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      const double prev = __shfl_up_sync(0xffffffffu, incl, 1);
      const double excl = lane == 0 ? 0.0 : prev;
      const double Z = __shfl_sync(0xffffffffu, incl, 31);
      int last_all = last;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) last_all = max(last_all, __shfl_xor_sync(0xffffffffu, last_all, o));
      if (!(Z > 0.0) && mode != 0) {
        if (lane == 0) s_chunk = -2;  // degenerate residual
      } else {
        const double th = u2 * Z;
        int found = -1;
        double rel = INFINITY;
        if (excl <= th && th < incl) {
          double cum = excl;
          for (int c = lo; c < hi; ++c) {
            if (th < cum + s_R[c]) {
              found = c;
              rel = th - cum;
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
  constexpr int kPer = kChunk / kDecThreads;  // 4 consecutive columns per thread
  const int x0 = chunk * kChunk + tid * kPer;
  float r[kPer];
  if (x0 + kPer <= V) {
    if (a.dt_t == TT_F32) {
      const float4 w = __ldg(reinterpret_cast<const float4*>(trow + size_t(x0) * 4));
      r[0] = w.x;
      r[1] = w.y;
      r[2] = w.z;
      r[3] = w.w;
    } else {
      const uint2 w = __ldg(reinterpret_cast<const uint2*>(trow + size_t(x0) * 2));
      r[0] = __uint_as_float(w.x << 16);
      r[1] = __uint_as_float(w.x & 0xffff0000u);
      r[2] = __uint_as_float(w.y << 16);
      r[3] = __uint_as_float(w.y & 0xffff0000u);
    }
  } else {
#pragma unroll
    for (int q = 0; q < kPer; ++q) r[q] = x0 + q < V ? load_dt(trow, a.dt_t, x0 + q) : 0.f;
  }
  float run = 0.f;
  int last_pos = -1;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int x = x0 + q;
    const float v = x < V ? r_of(x, r[q], mode) : 0.f;
    if (v > 0.f) last_pos = x;
    r[q] = v;
    run += v;
  }
  // block prefix: fp64 scan within each warp, warp totals scanned by warp 0
  double incl = double(run);
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  const double prev = __shfl_up_sync(0xffffffffu, incl, 1);
  double excl = lane == 0 ? 0.0 : prev;
  if (lane == 31) s_wtot[warp] = incl;
  __syncthreads();
  if (tid == 0) {  // warp bases in order, so that the intervals tile exactly
    double acc_w = 0.0;
    for (int w = 0; w < kWarps; ++w) {
      s_wpre[w] = acc_w;
      acc_w += s_wtot[w];
    }
  }
  __syncthreads();
  const double base = s_wpre[warp];
  incl += base;
  excl += base;
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
    atomicMax(&s_pick, pick);
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
cudaError_t launch_pdl(K kernel, const DecideArgs& args, unsigned grid, unsigned block,
                       cudaStream_t stream, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
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
  if (args.mode_transfer_only)
    return launch_pdl(transfer_kernel, args, unsigned(args.B), kDecThreads, stream, pdl);
  return launch_pdl(decide_kernel, args, unsigned(args.B), kDecThreads, stream, pdl);
}

cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  constexpr int kWarpsPerBlock = 4;
  prep_kernel<<<(args.B + kWarpsPerBlock - 1) / kWarpsPerBlock, 32 * kWarpsPerBlock, 0, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace tt
