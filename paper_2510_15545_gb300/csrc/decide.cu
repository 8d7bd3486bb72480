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

__device__ __forceinline__ F2 f2_neg(F2 a) { return {-a.hi, -a.lo}; }

// a * b as a normalised pair (the product's rounding error from a fused
// multiply-add).
__device__ __forceinline__ F2 f2_mul_f(F2 a, float b) {
  const float p = __fmul_rn(a.hi, b);
  const float e = fmaf(a.hi, b, -p);
  const float lo = fmaf(a.lo, b, e);
  const float hi = __fadd_rn(p, lo);
  return {hi, __fsub_rn(lo, __fsub_rn(hi, p))};
}

// Order of normalised pairs (hi = fl(hi + lo)): lexicographic, which is the
// order of their values. Intervals whose ends are the same pairs tile exactly.
__device__ __forceinline__ bool f2_lt(F2 a, F2 b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}
__device__ __forceinline__ bool f2_le(F2 a, F2 b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo <= b.lo);
}

__device__ __forceinline__ F2 shfl_up_f2(F2 v, int o, int width) {
  return {__shfl_up_sync(0xffffffffu, v.hi, o, width), __shfl_up_sync(0xffffffffu, v.lo, o, width)};
}
__device__ __forceinline__ F2 shfl_f2(F2 v, int src, int width) {
  return {__shfl_sync(0xffffffffu, v.hi, src, width), __shfl_sync(0xffffffffu, v.lo, src, width)};
}

// Max / compensated sum over groups of WIDTH lanes (the whole warp calls).
template <int WIDTH>
__device__ __forceinline__ float group_max(float v) {
#pragma unroll
  for (int o = WIDTH / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o, WIDTH));
  return v;
}
template <int WIDTH>
__device__ __forceinline__ F2 group_sum(F2 v) {
#pragma unroll
  for (int o = WIDTH / 2; o > 0; o >>= 1) {
    const F2 w = {__shfl_xor_sync(0xffffffffu, v.hi, o, WIDTH),
                  __shfl_xor_sync(0xffffffffu, v.lo, o, WIDTH)};
    v = f2_add(v, w);  // f2_add is commutative bit for bit: every lane ends equal
  }
  return v;
}

// Coarse level of the inverse CDF (Alg. 4): over chunk masses R(c), c in
// [0, nch), in column order, the chunk where the running sum first exceeds
// theta = u * Z, Z the total, and theta minus the mass before that chunk.
// WIDTH lanes (sublane sl) take lane-contiguous ranges of chunks. theta past
// the end by rounding gives the last chunk with mass and rel = +inf. Every lane
// of the warp calls; results are per group.
template <int WIDTH, class MassFn>
__device__ __forceinline__ void coarse_pick(const MassFn& R, int nch, int lane, float u, int& chunk,
                                            F2& rel, F2& Z) {
  const int sl = lane & (WIDTH - 1);
  const int per = (nch + WIDTH - 1) / WIDTH;
  const int lo = min(nch, sl * per), hi = min(nch, lo + per);
  F2 loc = {0.f, 0.f};
  int last = -1;
  for (int c = lo; c < hi; ++c) {
    const F2 r = R(c);
    loc = f2_add(loc, r);
    if (r.hi > 0.f) last = c;
  }
  F2 incl = loc;
#pragma unroll
  for (int o = 1; o < WIDTH; o <<= 1) {
    const F2 n = shfl_up_f2(incl, o, WIDTH);
    if (sl >= o) incl = f2_add(n, incl);
  }
  const F2 prev = shfl_up_f2(incl, 1, WIDTH);
  const F2 excl = sl == 0 ? F2{0.f, 0.f} : prev;
  Z = shfl_f2(incl, WIDTH - 1, WIDTH);
  const F2 th = f2_mul_f(Z, u);
  int found = -1;
  F2 r_rel = {INFINITY, 0.f};
  if (f2_le(excl, th) && f2_lt(th, incl)) {
    F2 cum = excl;
    for (int c = lo; c < hi; ++c) {
      const F2 r = R(c);
      const F2 nx = f2_add(cum, r);
      if (r.hi > 0.f && f2_lt(th, nx)) {
        found = c;
        r_rel = f2_add(th, f2_neg(cum));
        break;
      }
      cum = nx;
    }
    if (found < 0) found = last;  // rounding inside the range: its last chunk with mass
  }
  const unsigned grp = (0xffffffffu >> (32 - WIDTH)) << (lane & ~(WIDTH - 1));
  const unsigned hit = __ballot_sync(0xffffffffu, found >= 0) & grp;
  int la = last;
#pragma unroll
  for (int o = WIDTH / 2; o > 0; o >>= 1) la = max(la, __shfl_xor_sync(0xffffffffu, la, o, WIDTH));
  const int src = hit ? __ffs(hit) - 1 : (lane & ~(WIDTH - 1));
  const int fc = __shfl_sync(0xffffffffu, found, src);
  const F2 fr = shfl_f2(r_rel, src, 32);
  if (hit) {
    chunk = fc;
    rel = fr;
  } else {  // theta at the very top: the last chunk with mass
    chunk = la < 0 ? 0 : la;
    rel = {INFINITY, 0.f};
  }
}

// One CTA (16 warps) per request.
//  before the grid-dependency wait: checks of the caller's inputs, the map,
//    the scored logits and both uniforms of every position;
//  rows: one half-warp per row rebuilds the normaliser of each target row and
//    each mapped draft row from the row-pass partials;
//  accept test (one thread per position) and, for every candidate row, the
//    coarse level of its residual (one half-warp per row), side by side;
//  fine level: the whole CTA re-reads the chosen chunk of the accepted row.
__global__ void __launch_bounds__(kDecThreads) decide_kernel(DecideArgs a) {
  __shared__ int s_col[TT_MAX_M], s_map[TT_MAX_M], s_first[TT_MAX_M], s_qi[TT_MAX_M];
  __shared__ int s_task[TT_MAX_M];
  __shared__ float s_zt[TT_MAX_M], s_zd[TT_MAX_M], s_u[TT_MAX_M];
  __shared__ float s_p[TT_MAX_M], s_q[TT_MAX_M], s_DM[TT_MAX_M], s_DS[TT_MAX_M];
  __shared__ float s_u2[TT_MAX_M + 1], s_M[TT_MAX_M + 1], s_S[TT_MAX_M + 1];
  __shared__ int s_cchunk[TT_MAX_M + 1];
  __shared__ F2 s_crel[TT_MAX_M + 1];
  __shared__ unsigned char s_cmode[TT_MAX_M + 1];
  __shared__ F2 s_R[kMaxChunksPerRow];
  __shared__ F2 s_wtot[kWarps], s_wpre[kWarps + 1];
  __shared__ int s_dcol[TT_MAX_K];
  __shared__ int s_a, s_pick, s_last, s_nd, s_err, s_bad;

  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int half = lane >> 4, hl = lane & 15;
  const bool want_draft = a.full_q || a.q_hat_in == nullptr;
  const bool q_from_logits = a.q_hat_in == nullptr && a.draft_probs == nullptr;
  const bool draft_rows = q_from_logits || a.full_q;  // draft normalisers needed

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
  if (q_from_logits && k > TT_MAX_K) st |= TT_REQ_TOO_LONG;
  if (tid == 0) {
    s_a = m;
    s_pick = -1;
    s_last = -1;
    s_nd = 0;
    s_err = 0;
    s_bad = 0;
  }
  __syncthreads();
  // One round of loads: the caller's columns and, read before the wait, the
  // alignment's status and map (every CTA of the row pass between the two
  // grids waits for the alignment grid before it lets this grid start; they
  // are read through L2 only).
  int bad = 0;
  if (st == 0) {
    for (int j = tid; j < m; j += kDecThreads) {
      const int col = a.target_cols[t0 + j];
      s_col[j] = col;
      if (col < 0 || col >= a.t.V) bad |= 1;
      int i = j;
      if (want_draft) {
        i = __ldcg(a.map + t0 + j);
        if (i < 0 || i >= k) bad |= 2;
      }
      s_map[j] = i;
    }
    if (q_from_logits)
      for (int i = tid; i < k; i += kDecThreads) {
        const int col = a.draft_cols[d0 + i];
        s_dcol[i] = col;
        if (col < 0 || col >= a.d.V) bad |= 1;
      }
  }
  const int s_in = a.status_in ? __ldcg(a.status_in + b) : 0;
  if (bad) atomicOr(&s_bad, bad);
  __syncthreads();
  if (st == 0 && (s_bad & 1)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (s_in != 0) st = s_in;  // the alignment's verdict comes first
  if (st == 0 && (s_bad & 2)) st |= TT_REQ_ID_OUT_OF_RANGE;

  const uint64_t req = a.request_base + uint64_t(b);
  if (st == 0) {
    for (int j = tid; j <= m; j += kDecThreads) {
      s_u2[j] = float(philox_uniform(a.seed, uint64_t(j), 1, req));
      if (j == m) continue;
      int f = j;  // first position of this run of equal map entries
      if (want_draft)
        while (f > 0 && s_map[f - 1] == s_map[j]) --f;
      s_first[j] = f;
      s_u[j] = float(philox_uniform(a.seed, uint64_t(j), 0, req));
      s_zt[j] = load_checked(a, a.t, a.dt_t, int64_t(t0) + b + j, s_col[j]);
      // q of position j sits at s_q[s_qi[j]]: per position when given, per
      // run when transferred from the draft logits here
      s_qi[j] = q_from_logits ? f : j;
      if (a.q_hat_in) {
        s_q[j] = a.q_hat_in[t0 + j];
      } else if (a.draft_probs) {
        s_q[j] = a.draft_probs[int64_t(d0) + s_map[j]];
      }
      if (draft_rows && f == j) {
        s_task[atomicAdd(&s_nd, 1)] = j;
        if (q_from_logits)
          s_zd[j] = load_checked(a, a.d, a.dt_d, int64_t(d0) + s_map[j], s_dcol[s_map[j]]);
      }
    }
  }
  __syncthreads();

  // ------------------------------ results of the kernels before this one
  grid_dependency_wait();
  if (st != 0) {
    if (tid == 0) {
      const int e = (a.err && __ldcg(a.err) == a.epoch) ? __ldcg(a.err + 1) : 0;
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = e ? e : st;
    }
    return;
  }
  if (tid == 0 && a.err && __ldcg(a.err) == a.epoch) s_err = __ldcg(a.err + 1);

  // ------ row normalisers: target rows 0..m, then the first row of each run
  // of equal map entries (the copy rule reuses it); a half-warp per row
  int nonfinite = 0;
  const int n_tasks = m + 1 + s_nd;
  for (int base = 2 * warp; base < n_tasks; base += 2 * kWarps) {
    const int task = base + half;
    const bool valid = task < n_tasks;
    const bool tgt = task <= m;
    int j = 0;
    int64_t row = int64_t(t0) + b;
    const RowSet* R = &a.t;
    float z = 0.f;
    if (valid) {
      if (tgt) {
        j = task;
        row += j;
        if (j < m) z = s_zt[j];
      } else {
        j = s_task[task - (m + 1)];
        row = int64_t(d0) + s_map[j];
        R = &a.d;
        if (q_from_logits) z = s_zd[j];
      }
    }
    const int nch = valid ? R->nch : 0;
    const Partial* part = R->part + row * R->nch;
    const bool cached = nch <= 128;
    Partial c8[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int c = hl + 16 * i;
      c8[i] = (cached && c < nch) ? part[c] : Partial{-INFINITY, 0.f};
    }
    float lmx = -INFINITY;
    if (cached) {
#pragma unroll
      for (int i = 0; i < 8; ++i) lmx = fmaxf(lmx, c8[i].m);
    } else {
      for (int c = hl; c < nch; c += 16) lmx = fmaxf(lmx, part[c].m);
    }
    const float mx = group_max<16>(lmx);
    F2 acc = {0.f, 0.f};
    if (mx != -INFINITY) {
      if (cached) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if (c8[i].m != -INFINITY) acc = f2_add(acc, F2{c8[i].s * ex2_approx(c8[i].m - mx), 0.f});
      } else {
        for (int c = hl; c < nch; c += 16) {
          const Partial q = part[c];
          if (q.m != -INFINITY) acc = f2_add(acc, F2{q.s * ex2_approx(q.m - mx), 0.f});
        }
      }
    }
    const F2 Ssum = group_sum<16>(acc);
    const float S = __fadd_rn(Ssum.hi, Ssum.lo);
    if (valid && hl == 0) {
      if (tgt) {
        float M = mx, St = S;
        if (j < m) {  // add back the scored token's term, left out by the row pass
          const RowResult rr = with_token(mx, S, z, R->scale);
          M = rr.M;
          St = rr.S;
          const float ph = exp2_scaled(z, R->scale, M) * __frcp_rn(St);
          s_p[j] = ph;
          if (a.p_hat) a.p_hat[t0 + j] = ph;
        }
        if (!(St > 0.f) || !isfinite(St) || isnan(M)) nonfinite = 1;
        s_M[j] = M;
        s_S[j] = St;
        if (a.lse) a.lse[row] = (M + lg2_approx(St)) * 0.6931471805599453f;
      } else {
        if (!(S > 0.f) || !isfinite(S) || mx == -INFINITY) nonfinite = 1;
        s_DM[j] = mx;
        s_DS[j] = S;
        if (q_from_logits) s_q[j] = exp2_scaled(z, R->scale, mx) * __frcp_rn(S);
      }
    }
  }
  if (__syncthreads_or(nonfinite) || s_err) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = s_err ? s_err : TT_REQ_NOT_FINITE;
    }
    return;
  }

  // --------------------------- accept while u_j q_j < p_j (u < 1 exactly)
  for (int j = tid; j < m; j += kDecThreads) {
    const float qh = s_q[s_qi[j]];
    if (a.q_hat_out) a.q_hat_out[t0 + j] = qh;
    if (!(s_u[j] * qh < s_p[j])) atomicMin(&s_a, j);
  }

  const int nch = a.t.nch;
  const int V = a.t.V;
  const float scale_t = a.t.scale;
  // coarse level of every candidate row's residual, side by side with the
  // accept test: one-hot q puts r_t = max(0, p_j - q_j) on t_j and p elsewhere
  // (the row itself when that residual has no mass, and for the bonus row m)
  if (!a.full_q) {
    for (int base = 2 * warp; base <= m; base += 2 * kWarps) {
      const int j0 = base + half;
      const bool valid = j0 <= m;
      const int j = valid ? j0 : m;
      const Partial* part = a.t.part + (int64_t(t0) + b + j) * nch;
      const float Mj = s_M[j], invS = __frcp_rn(s_S[j]);
      const int ct = j < m ? s_col[j] / kChunk : -1;
      const float pj = j < m ? s_p[j] : 0.f;
      const float rt = j < m ? fmaxf(0.f, pj - s_q[s_qi[j]]) : 0.f;
      auto base_mass = [&](int c) -> float {
        const Partial P = part[c];
        return P.m == -INFINITY ? 0.f : P.s * ex2_approx(P.m - Mj) * invS;
      };
      // does the one-hot residual have mass?
      const int per = (nch + 15) / 16;
      const int lo = min(nch, hl * per), hi = min(nch, lo + per);
      bool pos = false;
      for (int c = lo; c < hi && !pos; ++c) pos = base_mass(c) > 0.f;
      const unsigned grp = 0xffffu << (lane & 16);
      const bool any = (__ballot_sync(0xffffffffu, pos) & grp) != 0;
      const int md = (j < m && (any || rt > 0.f)) ? 1 : 0;
      const float extra = j < m ? (md == 1 ? rt : pj) : 0.f;
      auto mass = [&](int c) -> F2 {
        F2 r = {base_mass(c), 0.f};
        if (c == ct) r = f2_add(r, F2{extra, 0.f});
        return r;
      };
      int chunk;
      F2 rel, Z;
      coarse_pick<16>(mass, nch, lane, s_u2[j], chunk, rel, Z);
      if (valid && hl == 0) {
        s_cchunk[j] = chunk;
        s_crel[j] = rel;
        s_cmode[j] = (unsigned char)md;
      }
    }
  }
  __syncthreads();
  const int acc = s_a;
  const int64_t row = int64_t(t0) + b + acc;
  const int col_t = acc < m ? s_col[acc] : -1;
  const float Mt = s_M[acc];
  const float invSt = __frcp_rn(s_S[acc]);
  const char* trow = a.t.data + row * a.t.stride_bytes;
  const float p_a = acc < m ? s_p[acc] : 0.f;
  const float r_t = acc < m ? fmaxf(0.f, p_a - s_q[s_qi[acc]]) : 0.f;
  const char* drow = nullptr;
  float Md = 0.f, invSd = 1.f;
  if (a.full_q && acc < m) {
    const int f = s_first[acc];
    drow = a.d.data + (int64_t(d0) + s_map[acc]) * a.d.stride_bytes;
    Md = s_DM[f];
    invSd = __frcp_rn(s_DS[f]);
  }
  // 0 the row itself, 1 one-hot residual, 2 full-q residual max(0, p - q)
  auto r_of = [&](int x, float z, int md) -> float {
    const float p = ex2_approx(fmaf(z, scale_t, -Mt)) * invSt;
    if (md == 1) return x == col_t ? r_t : p;
    if (md == 2) {
      const float q = ex2_approx(fmaf(load_dt(drow, a.dt_d, x), a.d.scale, -Md)) * invSd;
      return fmaxf(0.f, p - q);
    }
    return p;
  };
  if (a.full_q) {  // full-q residual: chunk masses from the logits themselves
    const Partial* part = a.t.part + row * nch;
    int md = acc < m ? 2 : 0;
    if (md == 2) {
      for (int c = warp; c < nch; c += kWarps) {
        F2 acc2 = {0.f, 0.f};
        const int hi_c = min(V, (c + 1) * kChunk);
        for (int x = c * kChunk + lane; x < hi_c; x += 32)
          acc2 = f2_add(acc2, F2{r_of(x, load_dt(trow, a.dt_t, x), 2), 0.f});
        const F2 Rc = group_sum<32>(acc2);
        if (lane == 0) s_R[c] = Rc;
      }
      __syncthreads();
    }
    if (warp == 0) {
      auto mass0 = [&](int c) -> F2 {
        const Partial P = part[c];
        F2 r = {P.m == -INFINITY ? 0.f : P.s * ex2_approx(P.m - Mt) * invSt, 0.f};
        if (col_t >= 0 && c == col_t / kChunk) r = f2_add(r, F2{p_a, 0.f});
        return r;
      };
      auto mass2 = [&](int c) -> F2 { return s_R[c]; };
      int chunk;
      F2 rel, Z;
      if (md == 2) {
        coarse_pick<32>(mass2, nch, lane, s_u2[acc], chunk, rel, Z);
        if (!(Z.hi > 0.f)) md = 0;  // degenerate residual: the row itself
      }
      if (md == 0) coarse_pick<32>(mass0, nch, lane, s_u2[acc], chunk, rel, Z);
      if (lane == 0) {
        s_cchunk[acc] = chunk;
        s_crel[acc] = rel;
        s_cmode[acc] = (unsigned char)md;
      }
    }
    __syncthreads();
  }
  const int chunk = s_cchunk[acc];
  const F2 rel = s_crel[acc];
  const int mode = s_cmode[acc];

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
  F2 run = {0.f, 0.f};
  int last_pos = -1;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int x = x0 + q;
    const float v = x < V ? r_of(x, r[q], mode) : 0.f;
    if (v > 0.f) last_pos = x;
    r[q] = v;
    run = f2_add(run, F2{v, 0.f});
  }
  // block prefix in pairs: scan within each warp, warp totals scanned by
  // warp 0; a warp's last interval ends where the next warp's first begins
  F2 incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const F2 n = shfl_up_f2(incl, o, 32);
    if (lane >= o) incl = f2_add(n, incl);
  }
  const F2 prev = shfl_up_f2(incl, 1, 32);
  F2 excl = lane == 0 ? F2{0.f, 0.f} : prev;
  if (lane == 31) s_wtot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const F2 t = lane < kWarps ? s_wtot[lane] : F2{0.f, 0.f};
    F2 wi = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const F2 n = shfl_up_f2(wi, o, 32);
      if (lane >= o) wi = f2_add(n, wi);
    }
    const F2 wp = shfl_up_f2(wi, 1, 32);
    if (lane <= kWarps) s_wpre[lane] = lane == 0 ? F2{0.f, 0.f} : wp;
  }
  __syncthreads();
  const F2 base = s_wpre[warp];
  incl = lane == 31 ? s_wpre[warp + 1] : f2_add(base, incl);
  excl = f2_add(base, excl);
  if (f2_le(excl, rel) && f2_lt(rel, incl)) {
    F2 c = excl;
    int pick = last_pos;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      c = f2_add(c, F2{r[q], 0.f});
      if (r[q] > 0.f && f2_lt(rel, c)) {
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
  if (a.work && blockIdx.x == 0 && threadIdx.x < kWorkShards)
    a.work[threadIdx.x * kWorkStride] = 0ull;  // read after this grid ends
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
