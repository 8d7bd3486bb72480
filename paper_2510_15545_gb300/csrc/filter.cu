// filter.cu -- verification under the sampling filters of the paper's
// generation hyperparameters (temperature, top-k, top-p), for the families
// whose rows the row pass reduced to top-k lists (one sorted list of k
// candidates per row unit: 2048 fp32 or 4096 bf16 columns).
//
// (Nucleus rows, top-p without top-k, are found in nucleus.cu; filter_q_kernel
// takes both kinds of draft rows.)
//
// A filtered row's distribution is fixed by its top k logits: kept_kernel
// merges the row's unit lists into its top-k (one warp per row, every
// filtered row of the call at once), then softmax at temperature, the top-p
// cut and renormalisation give the kept set, stored as k (probability,
// column) entries. filter_q_kernel turns the mapped draft rows' kept sets
// into q_hat (§4.2, App. A.2 with the filtered draft distribution);
// decide_filtered_kernel takes p_hat from the target rows' kept sets, runs
// the accept test (Alg. 2 / Alg. 4) and draws the next token from the
// residual (or the bonus row) over the kept set, in column order.
#include <algorithm>
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"
#include "tt_f2.cuh"

namespace tt {

namespace {

constexpr int kFThreads = 256;
constexpr int kFWarps = kFThreads / 32;
constexpr int kRowCap = 256;  // merge candidates of one row a warp keeps in shared memory

// Inclusive prefix in pairs over the warp's lanes.
__device__ __forceinline__ F2 warp_scan_f2(F2 v, int lane) {
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const F2 n = shfl_up_f2(v, o);
    if (lane >= o) v = f2_add(n, v);
  }
  return v;
}

__device__ __forceinline__ float load_logit_dt(const char* row, int dt, int64_t col) {
  return dt == TT_F32 ? load_logit<TT_F32>(row, col) : load_logit<TT_BF16>(row, col);
}

__device__ __forceinline__ bool cand_before(float v1, int c1, float v2, int c2) {
  return v1 > v2 || (v1 == v2 && c1 < c2);
}

// Warp-wide best element after (pv, pc) in candidate order; f = found.
__device__ __forceinline__ void warp_best(float& bv, int& bc, bool& f) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oc = __shfl_xor_sync(0xffffffffu, bc, o);
    const bool of = __shfl_xor_sync(0xffffffffu, int(f), o) != 0;
    if (of && (!f || cand_before(ov, oc, bv, bc))) {
      bv = ov;
      bc = oc;
      f = true;
    }
  }
}

constexpr int kMergeLists = 4;  // lists a lane owns in the K-way merge (rows of <= 128 units)

// The top-K of one filtered row by a K-way merge of its nch ordered unit
// lists: lane l owns lists l, l + 32, ... and keeps each one's current and
// next entry in registers; every round a warp-wide arg-best takes the winner
// and its owner advances that list, loading the entry after next. Exact, no
// candidate buffer. Rows of more than 32 * kMergeLists units use row_topk_wide.
__device__ void row_topk_merge(const Cand* lists, int nch, int K, int Ls, int lane, Cand* top) {
  Cand cur[kMergeLists], nxt[kMergeLists];
  int pos[kMergeLists];
#pragma unroll
  for (int i = 0; i < kMergeLists; ++i) {
    const int c = lane + 32 * i;
    const bool ok = c < nch;
    cur[i] = ok ? lists[int64_t(c) * Ls] : Cand{-INFINITY, -1};
    nxt[i] = ok && K > 1 ? lists[int64_t(c) * Ls + 1] : Cand{-INFINITY, -1};
    pos[i] = 1;  // index of nxt in its list
  }
  for (int r = 0; r < K; ++r) {
    // this lane's best current head
    float bv = -INFINITY;
    int bc = 0x7fffffff, bi = -1;
#pragma unroll
    for (int i = 0; i < kMergeLists; ++i)
      if (cur[i].c >= 0 && (bi < 0 || cand_before(cur[i].v, cur[i].c, bv, bc))) {
        bv = cur[i].v;
        bc = cur[i].c;
        bi = i;
      }
    bool f = bi >= 0;
    float wv = bv;
    int wc = bc;
    warp_best(wv, wc, f);
    if (lane == 0) top[r] = f ? Cand{wv, wc} : Cand{-INFINITY, -1};
    if (!f) continue;
    // the owner (columns are distinct) advances the winning list
    if (bi >= 0 && bc == wc && bv == wv) {
#pragma unroll
      for (int i = 0; i < kMergeLists; ++i)
        if (i == bi) {
          cur[i] = nxt[i];
          ++pos[i];
          const int c = lane + 32 * i;
          nxt[i] = pos[i] < K ? lists[int64_t(c) * Ls + pos[i]] : Cand{-INFINITY, -1};
        }
    }
  }
  __syncwarp();
}

// The top-K of one filtered row (its nch unit lists of K entries merged),
// ordered by cand_before, padded with (-inf, -1). One warp; `scr` holds
// kRowCap candidates, `top` K entries (shared memory). For rows of many units.
__device__ void row_topk_wide(const Cand* lists, int nch, int K, int Ls, int lane, Cand* scr,
                              Cand* top) {
  // tau: the K-th best list head (fewer than K heads: every entry counts)
  float tau = -INFINITY;
  {
    float pv = INFINITY;
    int pc = -1;
    for (int r = 0; r < K; ++r) {
      float bv = -INFINITY;
      int bc = 0x7fffffff;
      bool f = false;
      for (int c = lane; c < nch; c += 32) {
        const Cand h = lists[int64_t(c) * Ls];
        if (h.c >= 0 && cand_before(pv, pc, h.v, h.c) && (!f || cand_before(h.v, h.c, bv, bc))) {
          bv = h.v;
          bc = h.c;
          f = true;
        }
      }
      warp_best(bv, bc, f);
      if (!f) {
        tau = -INFINITY;
        break;
      }
      pv = bv;
      pc = bc;
      if (r == K - 1) tau = bv;
    }
  }
  // candidates: every list entry at or above tau (lists are ordered)
  int cnt = 0;
  for (int c = lane; c < nch; c += 32)
    for (int i = 0; i < K; ++i) {
      const Cand x = lists[int64_t(c) * Ls + i];
      if (x.c < 0 || x.v < tau) break;
      ++cnt;
    }
  int incl = cnt;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  const int C = __shfl_sync(0xffffffffu, incl, 31);
  if (C <= kRowCap) {
    int pos = incl - cnt;
    for (int c = lane; c < nch; c += 32)
      for (int i = 0; i < K; ++i) {
        const Cand x = lists[int64_t(c) * Ls + i];
        if (x.c < 0 || x.v < tau) break;
        scr[pos++] = x;
      }
    __syncwarp();
    for (int i = lane; i < C; i += 32) {
      const Cand ci = scr[i];
      int r = 0;
      for (int j = 0; j < C; ++j) r += cand_before(scr[j].v, scr[j].c, ci.v, ci.c);
      if (r < K) top[r] = ci;
    }
    for (int r = C + lane; r < K; r += 32) top[r] = Cand{-INFINITY, -1};
  } else {
    // exact extraction over every list entry
    float pv = INFINITY;
    int pc = -1;
    for (int r = 0; r < K; ++r) {
      float bv = -INFINITY;
      int bc = 0x7fffffff;
      bool f = false;
      for (int c = lane; c < nch; c += 32)
        for (int i = 0; i < K; ++i) {
          const Cand x = lists[int64_t(c) * Ls + i];
          if (x.c < 0) break;
          if (cand_before(pv, pc, x.v, x.c) && (!f || cand_before(x.v, x.c, bv, bc))) {
            bv = x.v;
            bc = x.c;
            f = true;
          }
        }
      warp_best(bv, bc, f);
      if (lane == 0) top[r] = f ? Cand{bv, bc} : Cand{-INFINITY, -1};
      if (f) {
        pv = bv;
        pc = bc;
      } else {
        pv = -INFINITY;
        pc = 0x7fffffff;
      }
    }
  }
  __syncwarp();
}

constexpr int kPre = 4;  // entries of each list loaded before the threshold is known
static_assert(kPre == 4, "the first entries are loaded as two 16-byte pairs");

// The top-K of one filtered row of nl <= 32 * kMergeLists unit lists, by a
// threshold. Lane l owns lists l, l + 32, ...; tau, the K-th largest of the
// 64 values formed by each lane's two largest first-or-second list entries,
// bounds the row's K-th largest from below (they are 64 distinct elements of
// the row, so K elements reach tau). Every list entry at or above tau is a candidate: the
// leading run of each list, usually a little over K entries in all. They are
// gathered in `scr` and ranked by counting; more than kRowCap (runs of equal
// logits) take the K-way merge instead.
__device__ void row_topk_thresh(const Cand* lists, int nl, int K, int Ls, int lane, Cand* scr,
                                Cand* top) {
  Cand e[kMergeLists][kPre];
  float m1 = -INFINITY, m2 = -INFINITY;  // the lane's two largest heads
  const Cand pad = {-INFINITY, -1};
#pragma unroll
  for (int i = 0; i < kMergeLists; ++i) {
    const int c = lane + 32 * i;
    // entries 0-3 as two 16-byte loads (a list starts on a 16-byte boundary
    // and holds an even number of slots; slots past K are not read)
    e[i][0] = e[i][1] = e[i][2] = e[i][3] = pad;
    if (c < nl) {
      const uint4* L = reinterpret_cast<const uint4*>(lists + int64_t(c) * Ls);
      const uint4 a = L[0];
      e[i][0] = Cand{__uint_as_float(a.x), int32_t(a.y)};
      if (K > 1) e[i][1] = Cand{__uint_as_float(a.z), int32_t(a.w)};
      if (K > 2) {
        const uint4 b = L[1];
        e[i][2] = Cand{__uint_as_float(b.x), int32_t(b.y)};
        if (K > 3) e[i][3] = Cand{__uint_as_float(b.z), int32_t(b.w)};
      }
    }
    // a list's first two entries are distinct elements: each lane offers the
    // two largest first-or-second entries of its lists
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const float h = e[i][j].c >= 0 ? e[i][j].v : -INFINITY;
      m2 = fmaxf(m2, fminf(m1, h));
      m1 = fmaxf(m1, h);
    }
  }
  // the 32 largest of the 64: half-cleaner of (m1 descending, m2 ascending)
  const float top32 =
      warp_merge_desc(fmaxf(warp_sort<true>(m1, lane), warp_sort<false>(m2, lane)), lane);
  const float tau = __shfl_sync(0xffffffffu, top32, K - 1);
  // leading run of each list at or above tau (entries past kPre read here)
  int cnt[kMergeLists];
  int nc = 0;
#pragma unroll
  for (int i = 0; i < kMergeLists; ++i) {
    const int c = lane + 32 * i;
    int k = 0;
#pragma unroll
    for (int j = 0; j < kPre; ++j) k += (k == j && e[i][j].c >= 0 && e[i][j].v >= tau) ? 1 : 0;
    if (k == kPre && c < nl) {
      // the run may go on: a list is ordered, so counting its entries at or
      // above tau gives the run's length, with independent loads
#pragma unroll 8
      for (int j = kPre; j < K; ++j) {
        const Cand x = lists[int64_t(c) * Ls + j];
        k += (x.c >= 0 && x.v >= tau) ? 1 : 0;
      }
    }
    cnt[i] = k;
    nc += k;
  }
  int incl = nc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += x;
  }
  const int C = __shfl_sync(0xffffffffu, incl, 31);
  if (C > kRowCap) {
    row_topk_merge(lists, nl, K, Ls, lane, top);
    return;
  }
  int p = incl - nc;
#pragma unroll
  for (int i = 0; i < kMergeLists; ++i) {
    const int c = lane + 32 * i;
#pragma unroll
    for (int j = 0; j < kPre; ++j)
      if (j < cnt[i]) scr[p++] = e[i][j];
#pragma unroll 4
    for (int j = kPre; j < cnt[i]; ++j) scr[p++] = lists[int64_t(c) * Ls + j];
  }
  __syncwarp();
  for (int i = lane; i < C; i += 32) {
    const Cand ci = scr[i];
    int r = 0;
#pragma unroll 4
    for (int j = 0; j < C; ++j) {
      const Cand cj = scr[j];
      r += cand_before(cj.v, cj.c, ci.v, ci.c);
    }
    if (r < K) top[r] = ci;
  }
  for (int r = C + lane; r < K; r += 32) top[r] = Cand{-INFINITY, -1};
  __syncwarp();
}

// The top-K of a row of at most 64 list entries (nl * K <= 64): every entry
// is a candidate, loaded one or two per lane. Entry s (place s % K of list
// s / K) comes after the s % K entries ahead of it in its own list (a list's
// real entries lead it) and after those entries of the other lists that
// cand_before puts first.
__device__ void row_topk_small(const Cand* lists, int nl, int K, int Ls, int lane, Cand* scr,
                               Cand* top) {
  const int n = nl * K;
  Cand x[2];
  int own[2], place[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int s = lane + 32 * h;
    own[h] = s / K;
    place[h] = s - own[h] * K;
    x[h] = s < n ? lists[int64_t(own[h]) * Ls + place[h]] : Cand{-INFINITY, -1};
    scr[s] = x[h];
  }
  __syncwarp();
  const int nvalid = __popc(__ballot_sync(0xffffffffu, x[0].c >= 0)) +
                     __popc(__ballot_sync(0xffffffffu, x[1].c >= 0));
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (x[h].c < 0) continue;
    int r = place[h];
    for (int l = 0; l < nl; ++l) {
      if (l == own[h]) continue;
#pragma unroll 4
      for (int j = 0; j < K; ++j) {
        const Cand y = scr[l * K + j];
        r += (y.c >= 0 && cand_before(y.v, y.c, x[h].v, x[h].c)) ? 1 : 0;
      }
    }
    if (r < K) top[r] = x[h];
  }
  for (int r = nvalid + lane; r < K; r += 32) top[r] = Cand{-INFINITY, -1};
  __syncwarp();
}

// The top-K of a row of two unit lists (a 4096-column fp32 row): the first K
// places of the merge of two ordered lists. Lane i finds by a binary search
// over the merge path how many of its first i places list A fills; the
// entries come from the two lists held one per lane and fetched by shuffles.
__device__ void row_topk_two(const Cand* lists, int K, int Ls, int lane, Cand* top) {
  const Cand pad = {-INFINITY, -1};
  const Cand A = lane < K ? lists[lane] : pad;
  const Cand Bv = lane < K ? lists[Ls + lane] : pad;
  // list entries past their real ones (pads) rank last
  auto a_at = [&](int x) -> Cand {
    const float v = __shfl_sync(0xffffffffu, A.v, x & 31);
    const int c = __shfl_sync(0xffffffffu, A.c, x & 31);
    return Cand{v, c};
  };
  auto b_at = [&](int x) -> Cand {
    const float v = __shfl_sync(0xffffffffu, Bv.v, x & 31);
    const int c = __shfl_sync(0xffffffffu, Bv.c, x & 31);
    return Cand{v, c};
  };
  auto before = [&](const Cand& x, const Cand& y) -> bool {  // x ranks before y
    if (x.c < 0) return false;
    if (y.c < 0) return true;
    return cand_before(x.v, x.c, y.v, y.c);
  };
  // place i: a = entries of A among the first i places (the merge path)
  const int i = lane;
  int lo = max(0, i - K), hi = min(i, K);
#pragma unroll 1
  for (int step = 0; step < 6; ++step) {  // lo < hi for at most log2(K) + 1 steps
    const int mid = (lo + hi + 1) >> 1;
    const bool active = lo < hi;
    // with mid entries of A taken, A[mid - 1] must rank before B[i - mid]
    const Cand am = a_at(mid - 1), bm = b_at(i - mid);
    if (active) {
      if (i - mid >= K || before(am, bm)) lo = mid;
      else hi = mid - 1;
    }
  }
  const int a = lo, b = i - a;
  const Cand ca = a_at(a), cb = b_at(b);
  const bool take_a = a < K && (b >= K || before(ca, cb));
  const Cand pick = take_a ? ca : cb;
  if (lane < K) top[lane] = (take_a ? a < K : b < K) && pick.c >= 0 ? pick : pad;
  __syncwarp();
}

__device__ __forceinline__ void row_topk(const Cand* lists, int nch, int K, int Ls, int lane,
                                         Cand* scr, Cand* top) {
  if (nch == 2) row_topk_two(lists, K, Ls, lane, top);
  else if (nch * K <= 64) row_topk_small(lists, nch, K, Ls, lane, scr, top);
  else if (nch <= 32 * kMergeLists) row_topk_thresh(lists, nch, K, Ls, lane, scr, top);
  else row_topk_wide(lists, nch, K, Ls, lane, scr, top);
}

// The top-K of a row under the repetition penalty: its lists' top-K (which
// leave out the request's penalized columns; -inf entries stand in for them)
// merged with those columns, each at the row's own value: penalized (z * theta
// for z < 0, else z / theta, fp32) when the column's first sequence position
// lies before the row's, raw otherwise. In place in `top`; one warp.
__device__ void penalize_top(const KeptArgs& a, const RowSet& S, int dt, bool tgt, int64_t row,
                             int K, int lane, Cand* scr, Cand* top) {
  const int32_t* off = tgt ? a.target_off : a.draft_off;
  int lo = 0, hi = a.B - 1;
  while (lo < hi) {  // the row's request: largest b whose first row is at or before row
    const int mid = (lo + hi + 1) >> 1;
    if (int64_t(off[mid]) + (tgt ? mid : 0) <= row) lo = mid;
    else hi = mid - 1;
  }
  const int b = lo;
  const int64_t j = row - (int64_t(off[b]) + (tgt ? b : 0));  // position of the row
  const int base = S.pbase[b], cnt = S.pcnt[b];
  const float th = S.penalty;
  const char* zrow = S.data + row * S.stride_bytes;
  const Cand me = lane < K ? top[lane] : Cand{-INFINITY, -1};
  const bool real = lane < K && me.c >= 0 && me.v > -INFINITY;
  const int nt = __popc(__ballot_sync(0xffffffffu, real));  // a prefix of the lanes
  const bool full = nt == K;
  const float tv = __shfl_sync(0xffffffffu, me.v, K - 1);
  const int tc = __shfl_sync(0xffffffffu, me.c, K - 1);
  auto value = [&](const PenEntry& e) -> float {
    const float z = load_logit_dt(zrow, dt, e.col);
    return e.first < j ? (z < 0.f ? __fmul_rn(z, th) : __fdiv_rn(z, th)) : z;
  };
  __syncwarp();
  if (real) scr[lane] = me;
  int n = nt;
  for (int i0 = 0; i0 < cnt; i0 += 32) {
    const int i = i0 + lane;
    Cand c = {-INFINITY, -1};
    bool q = false;
    if (i < cnt) {
      const PenEntry e = S.pen[base + i];
      c = Cand{value(e), e.col};
      q = c.v > -INFINITY && (!full || cand_before(c.v, c.c, tv, tc));
    }
    const unsigned m = __ballot_sync(0xffffffffu, q);
    const int pos = n + __popc(m & ((1u << lane) - 1u));
    if (q && pos < kRowCap) scr[pos] = c;
    n += __popc(m);
  }
  __syncwarp();
  if (n <= kRowCap) {
    for (int i = lane; i < n; i += 32) {
      const Cand ci = scr[i];
      int r = 0;
      for (int x = 0; x < n; ++x) r += cand_before(scr[x].v, scr[x].c, ci.v, ci.c);
      if (r < K) top[r] = ci;
    }
    for (int r = n + lane; r < K; r += 32) top[r] = Cand{-INFINITY, -1};
  } else {
    // more candidates than the buffer: K rounds of a warp arg-best over the
    // list entries and the penalized columns
    float pv = INFINITY;
    int pc = -1;
    for (int r = 0; r < K; ++r) {
      float bv = -INFINITY;
      int bc = 0x7fffffff;
      bool f = false;
      if (real && cand_before(pv, pc, me.v, me.c)) {
        bv = me.v;
        bc = me.c;
        f = true;
      }
      for (int i = lane; i < cnt; i += 32) {
        const PenEntry e = S.pen[base + i];
        const float v = value(e);
        if (v > -INFINITY && cand_before(pv, pc, v, e.col) && (!f || cand_before(v, e.col, bv, bc))) {
          bv = v;
          bc = e.col;
          f = true;
        }
      }
      warp_best(bv, bc, f);
      if (lane == 0) top[r] = f ? Cand{bv, bc} : Cand{-INFINITY, -1};
      if (f) {
        pv = bv;
        pc = bc;
      } else {
        pv = -INFINITY;
        pc = 0x7fffffff;
      }
    }
  }
  __syncwarp();
}

// The kept set of a filtered row from its top-K (in shared memory): lane i < n
// holds kept entry i (column, probability); returns n (0: no finite logit).
// lse = natural log of the kept set's normaliser sum exp(z / T).
__device__ int kept_set(const Cand* top, int K, float scale, float top_p, int lane, int& col,
                        float& prob, float& lse) {
  const Cand me = lane < K ? top[lane] : Cand{-INFINITY, -1};
  const float v0 = top[0].v;
  if (!(v0 > -INFINITY) || isnan(v0) || top[0].c < 0) {
    col = -1;
    prob = 0.f;
    lse = NAN;
    return 0;
  }
  const float M = __fmul_rn(v0, scale);
  const bool valid = lane < K && me.c >= 0;
  const float e = valid ? exp2_scaled(me.v, scale, M) : 0.f;
  const F2 incl = warp_scan_f2(F2{e, 0.f}, lane);
  const F2 all = {__shfl_sync(0xffffffffu, incl.hi, 31), __shfl_sync(0xffffffffu, incl.lo, 31)};
  const F2 prev = shfl_up_f2(incl, 1);
  const F2 before = lane == 0 ? F2{0.f, 0.f} : prev;
  // top-p: keep while the mass before the token is below top_p
  const bool keep = valid && (!(top_p < 1.f) || f2_lt(before, f2_mul_f(all, top_p)));
  const unsigned km = __ballot_sync(0xffffffffu, keep);
  const int n = __popc(km);  // a prefix of the lanes, so the kept sum is the prefix at n - 1
  const float S = __shfl_sync(0xffffffffu, __fadd_rn(incl.hi, incl.lo), n > 0 ? n - 1 : 0);
  col = keep ? me.c : -1;
  prob = keep ? e * __frcp_rn(S) : 0.f;
  lse = (M + lg2_approx(S)) * 0.6931471805599453f;
  return n;
}

// Probability of column c in the kept set held by the warp's lanes (0 if absent).
__device__ __forceinline__ float kept_prob(int col, float prob, int c) {
  const unsigned hit = __ballot_sync(0xffffffffu, col >= 0 && col == c);
  return hit ? __shfl_sync(0xffffffffu, prob, __ffs(hit) - 1) : 0.f;
}

// ------------------------------------------------------------ kept sets

// One warp per filtered row (draft rows first, then target rows; unneeded
// draft rows skipped): the row's top-K from its unit lists, then its kept set
// as K (probability, column) entries in value order, unused ones (0, -1),
// and the header (lse, kept count).
__global__ void __launch_bounds__(kFThreads, 4) kept_kernel(KeptArgs a) {
  __shared__ Cand s_scr[kFWarps][kRowCap];
  __shared__ Cand s_top[kFWarps][TT_MAX_TOP_K];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // (nucleus families' lists are read by the nucleus kernel)
  const int64_t rows_d = a.d.top_k > 0 && !a.d.nucleus ? a.rows_d : 0;
  const int64_t rows_t = a.t.top_k > 0 && !a.t.nucleus ? a.rows_t : 0;
  const int64_t total = rows_d + rows_t;
  const int64_t w0 = int64_t(blockIdx.x) * kFWarps + warp, stride = int64_t(gridDim.x) * kFWarps;
  grid_dependency_wait();  // the lists (and the need flags) come from earlier kernels
  // the next kernel reads only the caller's inputs before its own wait
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int64_t w = w0; w < total; w += stride) {
    const bool tgt = w >= rows_d;
    const int64_t row = tgt ? w - rows_d : w;
    const RowSet& S = tgt ? a.t : a.d;
    if (!tgt && S.need && S.need[row] == 0) continue;
    const int K = S.top_k;
    const int Ls = cand_stride(K);
    row_topk(S.cand + row * S.nlist * Ls, S.nlist, K, Ls, lane, s_scr[warp], s_top[warp]);
    if (S.pen) penalize_top(a, S, tgt ? a.dt_t : a.dt_d, tgt, row, K, lane, s_scr[warp],
                            s_top[warp]);
    int col;
    float prob, lse;
    const int n = kept_set(s_top[warp], K, S.scale, tgt ? a.top_p_t : a.top_p_d, lane, col,
                           prob, lse);
    Cand* out = (tgt ? a.kept_t : a.kept_d) + row * K;
    if (lane < K) out[lane] = Cand{col >= 0 ? prob : 0.f, col};
    if (lane == 0) (tgt ? a.head_t : a.head_d)[row] = KeptHead{lse, n};
  }
}

// A row's kept set as kept_set leaves it: lane l < K holds entry l.
__device__ __forceinline__ int load_kept(const Cand* kept, const KeptHead* head, int64_t row,
                                         int K, int lane, int& col, float& prob, float& lse) {
  const Cand e = lane < K ? kept[row * K + lane] : Cand{0.f, -1};
  col = e.c;
  prob = e.c >= 0 ? e.v : 0.f;
  const KeptHead h = head[row];
  lse = h.lse;
  return h.n;
}

// ------------------------------------------------------- q_hat, filtered

// NT threads per CTA: 256, or 128 when the batch has more requests than the
// GPU holds at once (more requests per SM, fewer threads idle at barriers).
template <int NT>
__global__ void __launch_bounds__(NT) filter_q_kernel(DecideArgs a) {
  constexpr int NW = NT / 32;
  __shared__ int s_map[TT_MAX_M];
  __shared__ float s_q[TT_MAX_M];
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int K = a.d.top_k;
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
  if (st == 0)
    for (int i = tid; i < k; i += NT) {
      const int col = a.draft_cols[d0 + i];
      if (col < 0 || col >= a.d.V) bad = 1;
    }
  grid_dependency_wait();
  if (st == 0)
    for (int j = tid; j < m; j += NT) {
      const int i = a.map[t0 + j];
      s_map[j] = i;
      if (i < 0 || i >= k) bad = 1;
    }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  if (st == 0 && a.status_p) st = a.status_p[b];  // the penalty's histories
  if (st == 0 && a.err && a.err[0] == a.epoch) st = a.err[1];
  if (st != 0) {
    if (!(st & (TT_REQ_BAD_OFFSETS | TT_REQ_TOO_LONG)))
      for (int j = tid; j < m; j += NT) a.q_hat_out[t0 + j] = 0.f;
    if (tid == 0) a.status[b] = st;
    return;
  }
  // one warp per run of equal map entries (the copy rule reuses its q)
  int nonfinite = 0;
  for (int j = warp; j < m; j += NW) {
    if (j > 0 && s_map[j] == s_map[j - 1]) continue;
    const int64_t row = int64_t(d0) + s_map[j];
    float q;
    if (a.d.nucleus) {  // kept when ranked at or before (tau, tau_col)
      const KeptHead h = a.head_d[row];
      if (h.n == 0) nonfinite = 1;
      const int c = a.draft_cols[row];
      const float z = load_logit_dt(a.d.data + row * a.d.stride_bytes, a.dt_d, c);
      const bool kept = z > h.tau || (z == h.tau && c <= h.tau_col);
      q = kept ? exp2_scaled(z, a.d.scale, h.M) * h.inv_s : 0.f;
    } else {
      int col;
      float prob, lse;
      const int n = load_kept(a.kept_d, a.head_d, row, K, lane, col, prob, lse);
      if (n == 0) nonfinite = 1;
      q = kept_prob(col, prob, a.draft_cols[row]);
    }
    if (lane == 0) s_q[j] = q;
  }
  const int nf = __syncthreads_or(nonfinite);
  for (int j = tid; j < m; j += NT) {
    int f = j;
    while (f > 0 && s_map[f - 1] == s_map[j]) --f;
    a.q_hat_out[t0 + j] = s_q[f];
  }
  if (tid == 0) a.status[b] = nf ? TT_REQ_NOT_FINITE : 0;
}

// ------------------------------------------------ decision, filtered target

template <int NT>
__global__ void __launch_bounds__(NT) decide_filtered_kernel(DecideArgs a) {
  constexpr int NW = NT / 32;
  __shared__ float s_p[TT_MAX_M];
  __shared__ int s_a, s_nf, s_pick;
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int K = a.t.top_k;
  int st = 0, t0 = 0, m = 0, d0 = 0, k = 0;
  if (!csr_ok(a.target_off, b, a.n_target) ||
      (a.full_q && !csr_ok(a.draft_off, b, a.n_draft))) {
    st = TT_REQ_BAD_OFFSETS;
  } else {
    t0 = a.target_off[b];
    m = a.target_off[b + 1] - t0;
    if (a.full_q) {
      d0 = a.draft_off[b];
      k = a.draft_off[b + 1] - d0;
    }
    if (m == 0 || (a.full_q && k == 0)) st |= TT_REQ_EMPTY;
    if (m > a.max_m || m > TT_MAX_M) st |= TT_REQ_TOO_LONG;
  }
  if (tid == 0) {
    s_a = m;
    s_nf = 0;
    s_pick = -1;
  }
  int bad = 0;
  if (st == 0)
    for (int j = tid; j < m; j += NT) {
      const int col = a.target_cols[t0 + j];
      if (col < 0 || col >= a.t.V) bad = 1;
    }
  if (__syncthreads_or(bad)) st |= TT_REQ_ID_OUT_OF_RANGE;
  grid_dependency_wait();
  if (a.status_in) {
    const int s_in = a.status_in[b];
    if (s_in != 0) st = s_in;  // the alignment's verdict comes first
  }
  if (st == 0 && a.status_q) st = a.status_q[b];  // then the transfer's
  if (st == 0 && a.status_p) st = a.status_p[b];  // then the penalty's histories
  if (a.err && a.err[0] == a.epoch) st = a.err[1];  // the row pass failed
  bad = 0;
  if (st == 0 && a.full_q)
    for (int j = tid; j < m; j += NT) {
      const int i = a.map[t0 + j];
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
  // target rows 0..m: kept sets, p_hat, lse; one warp per row
  for (int j = warp; j <= m; j += NW) {
    const int64_t row = int64_t(t0) + b + j;
    int col;
    float prob, lse;
    const int n = load_kept(a.kept_t, a.head_t, row, K, lane, col, prob, lse);
    if (n == 0 && lane == 0) s_nf = 1;
    if (j < m) {
      const float p = kept_prob(col, prob, a.target_cols[t0 + j]);
      if (lane == 0) {
        s_p[j] = p;
        if (a.p_hat) a.p_hat[t0 + j] = p;
      }
    }
    if (lane == 0 && a.lse) a.lse[row] = lse;
  }
  __syncthreads();
  if (s_nf) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = TT_REQ_NOT_FINITE;
    }
    return;
  }
  // accept while u_j q_j < p_j (u < 1 exactly)
  const uint64_t req = a.request_base + uint64_t(b);
  for (int j = tid; j < m; j += NT) {
    const float u = float(philox_uniform(a.seed, uint64_t(j), 0, req));
    if (!(u * a.q_hat_in[t0 + j] < s_p[j])) atomicMin(&s_a, j);
  }
  __syncthreads();
  const int acc = s_a;
  // the residual (or bonus) row acc over its kept set, in column order; warp 0
  if (warp == 0) {
    const int64_t row = int64_t(t0) + b + acc;
    int col;
    float prob, lse;
    load_kept(a.kept_t, a.head_t, row, K, lane, col, prob, lse);
    float qx = 0.f;  // what the residual takes away at this column
    if (acc < m) {
      if (a.full_q) {  // max(0, p - q) with the filtered draft row map[acc]
        const int64_t rd = int64_t(d0) + a.map[t0 + acc];
        int dcol;
        float dprob, dlse;
        load_kept(a.kept_d, a.head_d, rd, a.d.top_k, lane, dcol, dprob, dlse);
        // this lane's column in the draft's kept set (lanes hold distinct columns)
        float found = 0.f;
        for (int l = 0; l < 32; ++l) {
          const int c = __shfl_sync(0xffffffffu, dcol, l);
          const float pr = __shfl_sync(0xffffffffu, dprob, l);
          if (c >= 0 && c == col) found = pr;
        }
        qx = found;
      } else if (col >= 0 && col == a.target_cols[t0 + acc]) {
        qx = a.q_hat_in[t0 + acc];  // one-hot q
      }
    }
    float r = col >= 0 ? fmaxf(0.f, prob - qx) : 0.f;
    // total (pairs); no mass left: the row itself
    F2 z = warp_scan_f2(F2{r, 0.f}, lane);
    if (!(__shfl_sync(0xffffffffu, z.hi, 31) > 0.f)) r = col >= 0 ? prob : 0.f;
    // column order: this lane's rank among the kept columns
    int rank = 0;
    for (int l = 0; l < 32; ++l) {
      const int c = __shfl_sync(0xffffffffu, col, l);
      rank += c >= 0 && col >= 0 && c < col;
    }
    // gather the masses in column order: lane i takes the entry of rank i
    float rs = 0.f;
    int cs = -1;
    for (int l = 0; l < 32; ++l) {
      const int rk = __shfl_sync(0xffffffffu, rank, l);
      const int c = __shfl_sync(0xffffffffu, col, l);
      const float x = __shfl_sync(0xffffffffu, r, l);
      if (c >= 0 && rk == lane) {
        rs = x;
        cs = c;
      }
    }
    const F2 incl = warp_scan_f2(F2{rs, 0.f}, lane);
    const F2 Z = {__shfl_sync(0xffffffffu, incl.hi, 31), __shfl_sync(0xffffffffu, incl.lo, 31)};
    const float u2 = float(philox_uniform(a.seed, uint64_t(acc), 1, req));
    const F2 th = f2_mul_f(Z, u2);
    const F2 prev = shfl_up_f2(incl, 1);
    const F2 excl = lane == 0 ? F2{0.f, 0.f} : prev;
    // the first column whose running mass exceeds theta; rounding past the
    // end: the last column with mass
    const bool hit = cs >= 0 && rs > 0.f && !f2_lt(th, excl) && f2_lt(th, incl);
    const unsigned hm = __ballot_sync(0xffffffffu, hit);
    const unsigned pm = __ballot_sync(0xffffffffu, cs >= 0 && rs > 0.f);
    int pick = -1;
    if (hm) pick = __shfl_sync(0xffffffffu, cs, __ffs(hm) - 1);
    else if (pm) pick = __shfl_sync(0xffffffffu, cs, 31 - __clz(pm));
    if (lane == 0) s_pick = pick;
  }
  __syncthreads();
  if (tid == 0) {
    a.accepted[b] = acc;
    a.next_token[b] = s_pick;
    a.status[b] = s_pick >= 0 ? 0 : TT_REQ_NOT_FINITE;
  }
}

template <typename Kern>
cudaError_t launch_f(Kern kernel, int nt, const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (args.B == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(args.B));
  cfg.blockDim = dim3(nt);
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

cudaError_t preload_filter() {
  cudaFuncAttributes fa;
  cudaError_t e;
  if ((e = cudaFuncGetAttributes(&fa, kept_kernel)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, filter_q_kernel<128>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, filter_q_kernel<256>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&fa, decide_filtered_kernel<128>)) != cudaSuccess) return e;
  return cudaFuncGetAttributes(&fa, decide_filtered_kernel<256>);
}

cudaError_t launch_kept(const KeptArgs& args, cudaStream_t stream, int sm_count, bool pdl) {
  const int64_t rows = (args.d.top_k > 0 && !args.d.nucleus ? args.rows_d : 0) +
                       (args.t.top_k > 0 && !args.t.nucleus ? args.rows_t : 0);
  if (rows == 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((rows + kFWarps - 1) / kFWarps, int64_t(sm_count) * 8);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(blocks));
  cfg.blockDim = dim3(kFThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kept_kernel, args);
}

// 128 threads per request when the batch has more than four requests per SM
static bool f_small_ctas(const DecideArgs& a) { return int64_t(a.B) > int64_t(4) * a.sm_count; }

cudaError_t launch_filter_q(const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (f_small_ctas(args)) return launch_f(filter_q_kernel<128>, 128, args, stream, pdl);
  return launch_f(filter_q_kernel<256>, 256, args, stream, pdl);
}

cudaError_t launch_decide_filtered(const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (f_small_ctas(args)) return launch_f(decide_filtered_kernel<128>, 128, args, stream, pdl);
  return launch_f(decide_filtered_kernel<256>, 256, args, stream, pdl);
}

}  // namespace tt
