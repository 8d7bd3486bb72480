// decide.cu -- per-request decision of one verification step (§4.2, Alg. 2
// accept loop, Alg. 4 residual) and the standalone transfer (Alg. 2
// MapProbabilities, App. A.2).
//
// One CTA per request (256 threads, or 128 when the batch has more requests
// than fit on the GPU at once). From the row-pass partials it rebuilds the
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
#include "tt_f2.cuh"

namespace tt {

namespace {

constexpr int kDecThreads = 256;            // threads of the transfer kernel, most of a decision CTA
constexpr int kWarps = kDecThreads / 32;  // most warps of a decision CTA
constexpr int kDecSmemMax = 64 * 1024;  // largest dynamic shared memory of a decision CTA
// Dynamic shared memory up to which a decision CTA fits beside three row-pass
// CTAs on one SM (3 x 66 KB of the 228 KB, less per-CTA reservations).
constexpr int kDecSmemBeside = 24 * 1024;

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
// the next token run in compensated pairs (tt_f2.cuh).

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

__device__ __forceinline__ bool f2_le(F2 a, F2 b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo <= b.lo);
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

// Coarse level of the inverse CDF (Alg. 4). Chunk c in [0, nch) carries the
// mass base(c), plus `extra` on chunk ct (the scored token's chunk, or -1):
// extra = x_main when the masses then have a positive total, else x_alt (the
// residual falls back to the row itself). The chunk where the running sum,
// taken in column order, first exceeds theta = u * Z (Z the total) and theta
// minus the mass before it are returned; theta past the end by rounding gives
// the last chunk with mass and rel = +inf. WIDTH lanes (sublane sl) take
// lane-contiguous ranges of chunks. Every lane of the warp calls; results are
// per group of WIDTH lanes. The loops are kept rolled: this runs once per
// CTA, on an instruction cache that is usually cold, so code size is latency.
template <int WIDTH, class BaseFn>
__device__ __forceinline__ void coarse_pick(const BaseFn& base, int nch, int lane, float u, int ct,
                                            float x_main, float x_alt, int& chunk, F2& rel, F2& Z,
                                            bool& main_used) {
  const int sl = lane & (WIDTH - 1);
  const int per = (nch + WIDTH - 1) / WIDTH;
  const int lo = min(nch, sl * per), hi = min(nch, lo + per);
  const unsigned grp = (0xffffffffu >> (32 - WIDTH)) << (lane & ~(WIDTH - 1));
  F2 loc = {0.f, 0.f};
  int last = -1;
#pragma unroll 1
  for (int c = lo; c < hi; ++c) {
    const float r = base(c);
    loc = f2_add(loc, F2{r, 0.f});
    if (r > 0.f) last = c;
  }
  main_used = (__ballot_sync(0xffffffffu, last >= 0) & grp) != 0 || x_main > 0.f;
  const float extra = main_used ? x_main : x_alt;
  const bool own_ct = ct >= lo && ct < hi;
  if (own_ct) {
    loc = f2_add(loc, F2{extra, 0.f});
    if (extra > 0.f) last = max(last, ct);
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
#pragma unroll 1
    for (int c = lo; c < hi; ++c) {
      F2 r = {base(c), 0.f};
      if (c == ct) r = f2_add(r, F2{extra, 0.f});
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

// Shared memory of one decision CTA, sized by the batch's bounds: mx
// positions (max_m), kx draft columns (max_k, when q comes from the draft
// logits here) and nr chunk masses (full-q residual only).
struct DecSmem {
  F2* crel;      // [mx + 1] theta minus the mass before the coarse chunk, per candidate row
  F2* R;         // [nr] full-q residual chunk masses
  int* col;      // [mx] scored column of each target position
  int* map;      // [mx] i*(j)
  int* first;    // [mx] first position of each run of equal map entries
  int* qi;       // [mx] where q of position j sits in q
  int* task;     // [mx] first positions of the runs: the draft rows to normalise
  float* zt;     // [mx] scored target logits
  float* zd;     // [mx] scored draft logits (per run)
  float* u;      // [mx] accept uniforms
  float* p;      // [mx] p(t_j)
  float* q;      // [mx] q(t_j) (per position, or per run)
  float* DM;     // [mx] draft row maxima (per run)
  float* DS;     // [mx] draft row sums (per run)
  float* u2;     // [mx + 1] residual uniforms
  float* M;      // [mx + 1] target row maxima
  float* S;      // [mx + 1] target row sums
  int* cchunk;   // [mx + 1] coarse chunk per candidate row
  unsigned char* cmode;  // [mx + 1] residual mode per candidate row
  int* dcol;     // [kx] the request's draft columns
  size_t bytes;
};

__host__ __device__ inline DecSmem dec_smem(char* base, int mx, int kx, int nr) {
  DecSmem d;
  size_t off = 0;
  auto take = [&](size_t n) {
    char* r = base ? base + off : nullptr;
    off = (off + n + 15) & ~size_t(15);
    return r;
  };
  const size_t M1 = size_t(mx) + 1;
  d.crel = reinterpret_cast<F2*>(take(sizeof(F2) * M1));
  d.R = reinterpret_cast<F2*>(take(sizeof(F2) * size_t(nr)));
  d.col = reinterpret_cast<int*>(take(4 * size_t(mx)));
  d.map = reinterpret_cast<int*>(take(4 * size_t(mx)));
  d.first = reinterpret_cast<int*>(take(4 * size_t(mx)));
  d.qi = reinterpret_cast<int*>(take(4 * size_t(mx)));
  d.task = reinterpret_cast<int*>(take(4 * size_t(mx)));
  d.zt = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.zd = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.u = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.p = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.q = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.DM = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.DS = reinterpret_cast<float*>(take(4 * size_t(mx)));
  d.u2 = reinterpret_cast<float*>(take(4 * M1));
  d.M = reinterpret_cast<float*>(take(4 * M1));
  d.S = reinterpret_cast<float*>(take(4 * M1));
  d.cchunk = reinterpret_cast<int*>(take(4 * M1));
  d.cmode = reinterpret_cast<unsigned char*>(take(M1));
  d.dcol = reinterpret_cast<int*>(take(4 * size_t(kx)));
  d.bytes = off;
  return d;
}

__host__ __device__ inline int dec_kx(const DecideArgs& a) {
  const bool q_from_logits = a.q_hat_in == nullptr && a.draft_probs == nullptr;
  return q_from_logits ? min(max(a.max_k, 1), TT_MAX_K) : 0;
}
__host__ __device__ inline int dec_mx(const DecideArgs& a) {
  return min(max(a.max_m, 1), TT_MAX_M);
}
__host__ __device__ inline int dec_nr(const DecideArgs& a) { return a.full_q ? a.t.nch : 0; }

// Shared scalars of one decision CTA.
struct DecShared {
  F2 wtot[kWarps], wpre[kWarps + 1];
  int a, pick, last, nd, err;
};

// One CTA of NT threads (256, or 128 for batches larger than the GPU holds at
// once) per request.
//  before the grid-dependency wait: checks of the caller's inputs, the map,
//  the scored logits and both uniforms of every position;
//  after it: LPR lanes per row rebuild the normaliser of each target row and
//  each mapped draft row from the row-pass partials; the accept test and, for
//  every candidate row, the coarse level of its residual (LPR lanes per row)
//  run side by side; the whole CTA then re-reads the chosen chunk of the
//  accepted row (fine level).
// LPR is a power of two from 2 to 16, at least the row's chunk count where that
// is below 16, so that short rows do not leave most lanes of their group idle:
// 32 / LPR rows per warp.
// Small enough to sit beside the row pass's CTAs, so it starts while they
// stream: shared memory sized by the batch, and at most 56 registers, since
// registers come from each SM sub-partition's own file and one that holds 7
// row-pass warps (56 registers each) has room for 2 more such warps.
template <int NT, int LPR>
__global__ void __maxnreg__(56) decide_kernel(DecideArgs a) {
  constexpr int NW = NT / 32;  // warps of the CTA
  constexpr int G = 32 / LPR;  // row groups per warp
  static_assert(NW <= kWarps, "shared scan buffers hold kWarps warps");
  extern __shared__ __align__(16) char dsm[];
  __shared__ DecShared sh;
  __shared__ int s_bad;
  const int MX = dec_mx(a);
  const DecSmem sm = dec_smem(dsm, MX, dec_kx(a), dec_nr(a));

  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int grp = lane / LPR, hl = lane % LPR;
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
    if (m > a.max_m || m > MX) st |= TT_REQ_TOO_LONG;
  }
  if (q_from_logits && k > dec_kx(a)) st |= TT_REQ_TOO_LONG;
  if (tid == 0) {
    sh.a = m;
    sh.pick = -1;
    sh.last = -1;
    sh.nd = 0;
    sh.err = 0;
    s_bad = 0;
  }
  __syncthreads();
  // One round of loads: the caller's columns and, read before the wait, the
  // alignment's status and map (every CTA of the row pass between the two
  // grids waits for the alignment grid before it lets this grid start; they
  // are read through L2 only).
  int bad = 0;
  if (st == 0) {
    for (int j = tid; j < m; j += NT) {
      const int col = a.target_cols[t0 + j];
      sm.col[j] = col;
      if (col < 0 || col >= a.t.V) bad |= 1;
      int i = j;
      if (want_draft) {
        i = __ldcg(a.map + t0 + j);
        if (i < 0 || i >= k) bad |= 2;
      }
      sm.map[j] = i;
    }
    if (q_from_logits)
      for (int i = tid; i < k; i += NT) {
        const int col = a.draft_cols[d0 + i];
        sm.dcol[i] = col;
        if (col < 0 || col >= a.d.V) bad |= 1;
      }
  }
  const int s_in = a.status_in ? __ldcg(a.status_in + b) : 0;
  // (status_q, when given, comes from a kernel that ended before this grid started)
  const int s_q = a.status_q ? __ldcg(a.status_q + b) : 0;
  if (bad) atomicOr(&s_bad, bad);
  __syncthreads();
  if (st == 0 && (s_bad & 1)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st == 0 && s_q != 0) st = s_q;  // the transfer's verdict
  if (s_in != 0) st = s_in;  // the alignment's verdict comes first
  if (st == 0 && (s_bad & 2)) st |= TT_REQ_ID_OUT_OF_RANGE;

  const uint64_t req = a.request_base + uint64_t(b);
  if (st == 0) {
    for (int j = tid; j <= m; j += NT) {
      sm.u2[j] = float(philox_uniform(a.seed, uint64_t(j), 1, req));
      if (j == m) continue;
      int f = j;  // first position of this run of equal map entries
      if (want_draft)
        while (f > 0 && sm.map[f - 1] == sm.map[j]) --f;
      sm.first[j] = f;
      sm.u[j] = float(philox_uniform(a.seed, uint64_t(j), 0, req));
      sm.zt[j] = load_checked(a, a.t, a.dt_t, int64_t(t0) + b + j, sm.col[j]);
      // q of position j sits at q[qi[j]]: per position when given, per run
      // when transferred from the draft logits here
      sm.qi[j] = q_from_logits ? f : j;
      if (a.q_hat_in) {
        sm.q[j] = a.q_hat_in[t0 + j];
      } else if (a.draft_probs) {
        sm.q[j] = a.draft_probs[int64_t(d0) + sm.map[j]];
      }
      if (draft_rows && f == j) {
        sm.task[atomicAdd(&sh.nd, 1)] = j;
        if (q_from_logits)
          sm.zd[j] = load_checked(a, a.d, a.dt_d, int64_t(d0) + sm.map[j], sm.dcol[sm.map[j]]);
      }
    }
  }
  __syncthreads();

  // Pass 0 (dry) runs only in CTAs that start beside the row pass: it goes
  // through everything below on whatever the row-pass partials hold at the
  // time and writes nothing outside shared memory, so that this code is in the
  // SM's instruction cache when the real pass starts (one CTA per SM, on a
  // cold cache, spends more time fetching these instructions than running
  // them). Every index formed below stays in range whatever the values are.
  // Pass 1 starts at the grid-dependency wait.
#pragma unroll 1
  for (int pass = (st == 0 && int(blockIdx.x) < a.warm_ctas) ? 0 : 1; pass < 2; ++pass) {
    const bool dry = pass == 0;
    if (!dry) {
      __syncthreads();  // a dry pass is over everywhere
      // ---------------------------- results of the kernels before this one
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
      if (tid == 0) {  // read by others only past the rows phase's barrier
        sh.a = m;
        sh.pick = -1;
        sh.last = -1;
      }
    }
    // the row pass's error words: loaded now, looked at once the rows phase's
    // own loads are in flight
    int err0 = 0, err1 = 0;
    if (!dry && tid == 0 && a.err) {
      err0 = __ldcg(a.err);
      err1 = __ldcg(a.err + 1);
    }
    // ------ row normalisers: target rows 0..m, then the first row of each run
    // of equal map entries (the copy rule reuses it); LPR lanes per row
    int nonfinite = 0;
    const int n_tasks = m + 1 + sh.nd;
    for (int base = G * warp; base < n_tasks; base += G * NW) {
      const int task = base + grp;
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
          if (j < m) z = sm.zt[j];
        } else {
          j = sm.task[task - (m + 1)];
          row = int64_t(d0) + sm.map[j];
          R = &a.d;
          if (q_from_logits) z = sm.zd[j];
        }
      }
      const int nch = valid ? R->nch : 0;
      const Partial* part = R->part + row * R->nch;
      constexpr int kCache = LPR >= 8 ? 8 : 4;  // partials per lane held in registers
      const bool cached = nch <= kCache * LPR;
      Partial c8[kCache];
  #pragma unroll
      for (int i = 0; i < kCache; ++i) {
        const int c = hl + LPR * i;
        c8[i] = (cached && c < nch) ? part[c] : Partial{-INFINITY, 0.f};
      }
      float lmx = -INFINITY;
      if (cached) {
  #pragma unroll
        for (int i = 0; i < kCache; ++i) lmx = fmaxf(lmx, c8[i].m);
      } else {
        for (int c = hl; c < nch; c += LPR) lmx = fmaxf(lmx, part[c].m);
      }
      const float mx = group_max<LPR>(lmx);
      F2 acc = {0.f, 0.f};
      if (mx != -INFINITY) {
        if (cached) {
  #pragma unroll
          for (int i = 0; i < kCache; ++i)
            if (c8[i].m != -INFINITY) acc = f2_add(acc, F2{c8[i].s * ex2_approx(c8[i].m - mx), 0.f});
        } else {
          for (int c = hl; c < nch; c += LPR) {
            const Partial q = part[c];
            if (q.m != -INFINITY) acc = f2_add(acc, F2{q.s * ex2_approx(q.m - mx), 0.f});
          }
        }
      }
      const F2 Ssum = group_sum<LPR>(acc);
      const float S = __fadd_rn(Ssum.hi, Ssum.lo);
      if (valid && hl == 0) {
        if (tgt) {
          float M = mx, St = S;
          if (j < m) {  // add back the scored token's term, left out by the row pass
            const RowResult rr = with_token(mx, S, z, R->scale);
            M = rr.M;
            St = rr.S;
            const float ph = exp2_scaled(z, R->scale, M) * __frcp_rn(St);
            sm.p[j] = ph;
            if (a.p_hat && !dry) a.p_hat[t0 + j] = ph;
          }
          if (!(St > 0.f) || !isfinite(St) || isnan(M)) nonfinite = 1;
          sm.M[j] = M;
          sm.S[j] = St;
          if (a.lse && !dry) a.lse[row] = (M + lg2_approx(St)) * 0.6931471805599453f;
        } else {
          if (!(S > 0.f) || !isfinite(S) || mx == -INFINITY) nonfinite = 1;
          sm.DM[j] = mx;
          sm.DS[j] = S;
          if (q_from_logits) sm.q[j] = exp2_scaled(z, R->scale, mx) * __frcp_rn(S);
        }
      }
    }
    if (!dry && tid == 0 && a.err && err0 == a.epoch) sh.err = err1;
    if ((__syncthreads_or(nonfinite) || sh.err) && !dry) {
      if (tid == 0) {
        a.accepted[b] = 0;
        a.next_token[b] = -1;
        a.status[b] = sh.err ? sh.err : TT_REQ_NOT_FINITE;
      }
      return;
    }

    // --------------------------- accept while u_j q_j < p_j (u < 1 exactly)
    for (int j = tid; j < m; j += NT) {
      const float qh = sm.q[sm.qi[j]];
      if (a.q_hat_out && !dry) a.q_hat_out[t0 + j] = qh;
      if (!(sm.u[j] * qh < sm.p[j])) atomicMin(&sh.a, j);
    }

    const int nch = a.t.nch;
    const int V = a.t.V;
    const float scale_t = a.t.scale;
    // coarse level of every candidate row's residual, side by side with the
    // accept test: one-hot q puts r_t = max(0, p_j - q_j) on t_j and p elsewhere
    // (the row itself when that residual has no mass, and for the bonus row m)
    if (!a.full_q) {
      for (int base = G * warp; base <= m; base += G * NW) {
        const int j0 = base + grp;
        const bool valid = j0 <= m;
        const int j = valid ? j0 : m;
        const int64_t row = int64_t(t0) + b + j;
        const Partial* part = a.t.part + row * nch;
        const float Mj = sm.M[j], invS = __frcp_rn(sm.S[j]);
        const int ct = j < m ? sm.col[j] / kChunk : -1;
        const float pj = j < m ? sm.p[j] : 0.f;
        const float rt = j < m ? fmaxf(0.f, pj - sm.q[sm.qi[j]]) : 0.f;
        auto base_mass = [&](int c) -> float {
          const Partial P = part[c];
          return P.m == -INFINITY ? 0.f : P.s * ex2_approx(P.m - Mj) * invS;
        };
        int chunk;
        F2 rel, Z;
        bool main_used;
        coarse_pick<LPR>(base_mass, nch, lane, sm.u2[j], ct, rt, pj, chunk, rel, Z, main_used);
        if (valid && hl == 0) {
          sm.cchunk[j] = chunk;
          sm.crel[j] = rel;
          sm.cmode[j] = (unsigned char)(j < m && main_used ? 1 : 0);
        }
      }
    }
    __syncthreads();
    const int acc = sh.a;
    const int64_t row = int64_t(t0) + b + acc;
    const int col_t = acc < m ? sm.col[acc] : -1;
    const float Mt = sm.M[acc];
    const float invSt = __frcp_rn(sm.S[acc]);
    const char* trow = a.t.data + row * a.t.stride_bytes;
    const float p_a = acc < m ? sm.p[acc] : 0.f;
    const float r_t = acc < m ? fmaxf(0.f, p_a - sm.q[sm.qi[acc]]) : 0.f;
    const char* drow = nullptr;
    float Md = 0.f, invSd = 1.f;
    if (a.full_q && acc < m) {
      const int f = sm.first[acc];
      drow = a.d.data + (int64_t(d0) + sm.map[acc]) * a.d.stride_bytes;
      Md = sm.DM[f];
      invSd = __frcp_rn(sm.DS[f]);
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
        for (int c = warp; c < nch; c += NW) {
          F2 acc2 = {0.f, 0.f};
          const int hi_c = min(V, (c + 1) * kChunk);
          for (int x = c * kChunk + lane; x < hi_c; x += 32)
            acc2 = f2_add(acc2, F2{r_of(x, load_dt(trow, a.dt_t, x), 2), 0.f});
          const F2 Rc = group_sum<32>(acc2);
          if (lane == 0) sm.R[c] = Rc;
        }
        __syncthreads();
      }
      if (warp == 0) {
        auto mass0 = [&](int c) -> float {
          const Partial P = part[c];
          return P.m == -INFINITY ? 0.f : P.s * ex2_approx(P.m - Mt) * invSt;
        };
        auto mass2 = [&](int c) -> float { return __fadd_rn(sm.R[c].hi, sm.R[c].lo); };
        int chunk;
        F2 rel, Z;
        bool main_used;
        if (md == 2) {
          coarse_pick<32>(mass2, nch, lane, sm.u2[acc], -1, 0.f, 0.f, chunk, rel, Z, main_used);
          if (!(Z.hi > 0.f)) md = 0;  // degenerate residual: the row itself
        }
        if (md == 0)
          coarse_pick<32>(mass0, nch, lane, sm.u2[acc], col_t >= 0 ? col_t / kChunk : -1, p_a,
                          p_a, chunk, rel, Z, main_used);
        if (lane == 0) {
          sm.cchunk[acc] = chunk;
          sm.crel[acc] = rel;
          sm.cmode[acc] = (unsigned char)md;
        }
      }
      __syncthreads();
    }
    const int chunk = sm.cchunk[acc];
    const F2 rel = sm.crel[acc];
    const int mode = sm.cmode[acc];

    // ------------------------------------------ fine level: one chunk re-read,
    // in slabs of NT x 8 consecutive columns (8 per thread) taken in column
    // order; each slab is scanned as a block prefix in pairs, and the draw
    // minus the mass of the slabs before it is looked for in the next one
    constexpr int kPer = 8;
    constexpr int kSlabs = kChunk / (NT * kPer);
    F2 rel_s = rel;  // the draw relative to the current slab's start
#pragma unroll 1
    for (int slab = 0; slab < kSlabs; ++slab) {
      const int x0 = chunk * kChunk + slab * NT * kPer + tid * kPer;
      float r[kPer];
      if (x0 + kPer <= V) {
        if (a.dt_t == TT_F32) {
          const float4 w0 = __ldg(reinterpret_cast<const float4*>(trow + size_t(x0) * 4));
          const float4 w1 = __ldg(reinterpret_cast<const float4*>(trow + size_t(x0) * 4 + 16));
          r[0] = w0.x;
          r[1] = w0.y;
          r[2] = w0.z;
          r[3] = w0.w;
          r[4] = w1.x;
          r[5] = w1.y;
          r[6] = w1.z;
          r[7] = w1.w;
        } else {
          const uint4 w = __ldg(reinterpret_cast<const uint4*>(trow + size_t(x0) * 2));
          const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
    #pragma unroll
          for (int q = 0; q < 4; ++q) {
            r[2 * q] = __uint_as_float(ww[q] << 16);
            r[2 * q + 1] = __uint_as_float(ww[q] & 0xffff0000u);
          }
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
      if (lane == 31) sh.wtot[warp] = incl;
      __syncthreads();
      if (warp == 0) {
        const F2 t = lane < NW ? sh.wtot[lane] : F2{0.f, 0.f};
        F2 wi = t;
    #pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const F2 n = shfl_up_f2(wi, o, 32);
          if (lane >= o) wi = f2_add(n, wi);
        }
        const F2 wp = shfl_up_f2(wi, 1, 32);
        if (lane <= NW) sh.wpre[lane] = lane == 0 ? F2{0.f, 0.f} : wp;
      }
      __syncthreads();
      const F2 base = sh.wpre[warp];
      const F2 slab_total = sh.wpre[NW];
      incl = lane == 31 ? sh.wpre[warp + 1] : f2_add(base, incl);
      excl = f2_add(base, excl);
      if (f2_le(excl, rel_s) && f2_lt(rel_s, incl)) {
        F2 c = excl;
        int pick = last_pos;
    #pragma unroll
        for (int q = 0; q < kPer; ++q) {
          c = f2_add(c, F2{r[q], 0.f});
          if (r[q] > 0.f && f2_lt(rel_s, c)) {
            pick = x0 + q;
            break;
          }
        }
        atomicMax(&sh.pick, pick);
      }
      if (last_pos >= 0) atomicMax(&sh.last, last_pos);
      __syncthreads();
      if (sh.pick >= 0) break;  // the same for every thread (read past the barrier)
      rel_s = f2_add(rel_s, f2_neg(slab_total));
    }
    if (tid == 0 && !dry) {
      a.accepted[b] = acc;
      a.next_token[b] = sh.pick >= 0 ? sh.pick : sh.last;
      a.status[b] = 0;
    }
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
                       size_t smem, cudaStream_t stream, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args);
}

// Lanes per row of the decision kernel: the smallest power of two from 2 to 16
// that covers the chunks of every row it normalises.
int decide_lpr(const DecideArgs& a) {
  const bool draft_rows = (a.q_hat_in == nullptr && a.draft_probs == nullptr) || a.full_q;
  const int nch = draft_rows ? max(a.t.nch, a.d.nch) : a.t.nch;
  int l = 2;
  while (l < 16 && l < nch) l *= 2;
  return l;
}

template <int NT, int LPR>
cudaError_t preload_decide_variant() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, decide_kernel<NT, LPR>)) != cudaSuccess) return e;
  if ((e = cudaFuncSetAttribute(decide_kernel<NT, LPR>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, kDecSmemMax)) !=
      cudaSuccess)
    return e;
  // the same shared-memory split as the row pass, so that CTAs of both fit on one SM
  return cudaFuncSetAttribute(decide_kernel<NT, LPR>,
                              cudaFuncAttributePreferredSharedMemoryCarveout,
                              int(cudaSharedmemCarveoutMaxShared));
}

template <int NT>
cudaError_t preload_decide_nt() {
  cudaError_t e;
  if ((e = preload_decide_variant<NT, 2>()) != cudaSuccess) return e;
  if ((e = preload_decide_variant<NT, 4>()) != cudaSuccess) return e;
  if ((e = preload_decide_variant<NT, 8>()) != cudaSuccess) return e;
  return preload_decide_variant<NT, 16>();
}

template <int NT>
cudaError_t launch_decide_nt(const DecideArgs& a, size_t smem, cudaStream_t stream, bool pdl) {
  switch (decide_lpr(a)) {
    case 2: return launch_pdl(decide_kernel<NT, 2>, a, unsigned(a.B), NT, smem, stream, pdl);
    case 4: return launch_pdl(decide_kernel<NT, 4>, a, unsigned(a.B), NT, smem, stream, pdl);
    case 8: return launch_pdl(decide_kernel<NT, 8>, a, unsigned(a.B), NT, smem, stream, pdl);
    default: return launch_pdl(decide_kernel<NT, 16>, a, unsigned(a.B), NT, smem, stream, pdl);
  }
}

}  // namespace

cudaError_t preload_decide() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = preload_decide_nt<128>()) != cudaSuccess) return e;
  if ((e = preload_decide_nt<256>()) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, transfer_kernel)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, prep_kernel);
}

cudaError_t launch_decide(const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (args.B == 0) return cudaSuccess;
  if (args.mode_transfer_only)
    return launch_pdl(transfer_kernel, args, unsigned(args.B), kDecThreads, 0, stream, pdl);
  const size_t smem = dec_smem(nullptr, dec_mx(args), dec_kx(args), dec_nr(args)).bytes;
  if (smem > size_t(kDecSmemMax)) return cudaErrorInvalidConfiguration;
  DecideArgs a = args;
  // a warming pass is free only for CTAs that start beside the row pass
  if (!pdl || smem > size_t(kDecSmemBeside)) a.warm_ctas = 0;
  // 256 threads while the batch's CTAs all fit on the GPU at once (four per
  // SM: 56 registers x 256 threads), else 128 (nine per SM), which keeps more
  // requests in flight and fewer threads waiting at the CTA's barriers
  if (int64_t(a.B) > int64_t(4) * a.sm_count) return launch_decide_nt<128>(a, smem, stream, pdl);
  return launch_decide_nt<256>(a, smem, stream, pdl);
}

cudaError_t launch_prep(const PrepArgs& args, cudaStream_t stream) {
  if (args.B == 0) return cudaSuccess;
  constexpr int kWarpsPerBlock = 4;
  prep_kernel<<<(args.B + kWarpsPerBlock - 1) / kWarpsPerBlock, 32 * kWarpsPerBlock, 0, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace tt
