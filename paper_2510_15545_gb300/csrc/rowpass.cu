// rowpass.cu -- one streaming pass over logits rows: per chunk of kChunk
// columns, the maximum m of s_x = z_x * log2(e) / T and the sum of 2^(s_x - m).
//
// These partials are all the softmax normalisers of Alg. 2 / Alg. 4 need
// (log2 sum_x 2^s_x = M + log2 sum_c s_c 2^(m_c - M)) and they are the coarse
// level of the residual's inverse CDF, so every logit is read from HBM once.
// Target row j < m leaves its scored token t_j out of the sum; the decision
// kernel adds that one term back exactly. Draft rows that no target position
// maps to are skipped.
//
// Warp-specialised pipeline, several CTAs per SM: one producer lane streams
// chunks into a ring of shared-memory stages with 1-D bulk copies
// (cp.async.bulk, completion counted on an mbarrier per stage); each of the 8
// consumer warps owns every 8th stage, reduces one whole chunk at a time from
// shared memory (no block barrier) and frees the stage. Every wait is bounded in time; on timeout the kernel sets
// an error word that the decision kernel turns into a per-request status.
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstdlib>

#include "tt_device.cuh"
#include "tt_launch.h"
#include "tt_f2.cuh"

namespace tt {

namespace {

constexpr int kConsumerWarps = 8;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kRingBytes = 64 * 1024;  // three CTAs per SM fit
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr int kGrabMinBytes = 16 * 1024;   // smallest draw from the work counter
constexpr int kGrabMaxBytes = 128 * 1024;  // largest draw

// One stage holds one unit: cps consecutive chunks of one row (cps = 1 for
// fp32 rows, 2 for bf16 rows, so that every stage is one 8 KB bulk copy).
struct Desc {
  int64_t row;    // < 0: no more work for this consumer warp
  int32_t chunk;  // first chunk of the unit
  int32_t n;      // columns in the unit
  int32_t n_smem; // leading columns delivered by the bulk copy (rest read directly)
  int32_t excl;   // column (within the unit) left out of the sum, -1 = none
  int32_t set;    // 0 draft rows, 1 target rows
  int32_t req;    // the row's request when its family has a repetition penalty, else -1
};

// Stage s is always refilled for the same consumer warp (s mod kConsumerWarps),
// so a warp never waits on a stage more than one phase ahead of it: an
// mbarrier parity wait cannot tell phase n from phase n + 2.
constexpr int kCandCap = 128;   // top-k candidates of one unit a warp keeps in shared memory
constexpr int kDirectCap = 32;  // vectors at or above tau1 taken directly (more: tau2)
constexpr int kLevel2Cap = 64;  // vector maxima ranked by counting (more: radix search)

template <int DTD, int DTT, int SEL>
struct Ring {
  static constexpr int kStageBytes = kChunk * 4;  // one fp32 chunk or two bf16 chunks
  static constexpr int kCpsD = DTD == TT_F32 ? 1 : 2;  // chunks per stage, draft rows
  static constexpr int kCpsT = DTT == TT_F32 ? 1 : 2;  // chunks per stage, target rows
  static constexpr int kStages = kRingBytes / kStageBytes;
  static constexpr size_t kScratch = SEL ? size_t(kConsumerWarps) * kCandCap * sizeof(Cand) : 0;
  static constexpr size_t kSmem =
      size_t(kRingBytes) + kStages * (2 * sizeof(uint64_t) + sizeof(Desc)) + kScratch;
  static_assert(kStages % kConsumerWarps == 0, "each stage belongs to one consumer warp");
  static constexpr int kGrabMin = kGrabMinBytes / kStageBytes > 0 ? kGrabMinBytes / kStageBytes : 1;
  static constexpr int kGrabMax = kGrabMaxBytes / kStageBytes;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Waits for the phase of the given parity to complete; false after limit_ns.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          const uint64_t& limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1; i < (1u << 30); ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63) == 0 && global_ns() - t0 > limit_ns) return false;
  }
  return false;
}
__device__ __forceinline__ void bulk_copy_g2s(void* dst, const void* src, uint32_t bytes,
                                              uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void grid_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The scored columns of target rows visited mostly in increasing order: the
// request of the last row looked up is kept, so that the next row of the same
// request, or the first row of the next request, needs no search. The
// producer keeps it in shared memory, off its register budget.
struct ExclCursor {
  int b;           // request of the cached range (-1: none)
  int t0;          // its first target position
  int64_t r0, r1;  // its rows: r0 .. r1 (r1 is the bonus row)
};

__device__ __forceinline__ int excl_lookup(const RowPassArgs& a, ExclCursor* cur, int64_t r) {
  if (!a.target_off || a.B <= 0) return -1;
  int b = cur->b;
  if (!(b >= 0 && r >= cur->r0 && r <= cur->r1)) {
    if (b >= 0 && r == cur->r1 + 1 && b + 1 < a.B) {
      ++b;
    } else {
      int lo = 0, hi = a.B - 1;
      while (lo < hi) {  // largest b with target_off[b] + b <= r
        const int mid = (lo + hi + 1) >> 1;
        if (int64_t(a.target_off[mid]) + mid <= r) lo = mid;
        else hi = mid - 1;
      }
      b = lo;
    }
    const int t0 = a.target_off[b], t1 = a.target_off[b + 1];
    if (t0 < 0 || t1 < t0 || t1 > a.n_target) {
      cur->b = -1;
      return -1;
    }
    cur->b = b;
    cur->t0 = t0;
    cur->r0 = int64_t(t0) + b;
    cur->r1 = int64_t(t1) + b;
  }
  const int64_t j = r - cur->r0;
  if (j < 0 || j >= cur->r1 - cur->r0) return -1;  // the bonus row
  const int c = a.target_cols[cur->t0 + j];
  return (c >= 0 && c < a.t.V) ? c : -1;
}

// The request of a row, for rows visited mostly in increasing order (kept in
// shared memory like ExclCursor): target rows of request b are
// target_off[b] + b .. target_off[b+1] + b, draft rows draft_off[b] ..
// draft_off[b+1] - 1. -1 outside every request.
struct ReqCursor {
  int b;
  int64_t r0, r1;  // rows of request b: r0 .. r1 inclusive
};

__device__ __forceinline__ int req_lookup(const int32_t* off, int B, bool tgt, ReqCursor* cur,
                                          int64_t r) {
  if (!off || B <= 0) return -1;
  int b = cur->b;
  if (b >= 0 && r >= cur->r0 && r <= cur->r1) return b;
  if (b >= 0 && r == cur->r1 + 1 && b + 1 < B) {
    ++b;
  } else {
    int lo = 0, hi = B - 1;
    while (lo < hi) {  // largest b whose first row is at or before r
      const int mid = (lo + hi + 1) >> 1;
      if (int64_t(off[mid]) + (tgt ? mid : 0) <= r) lo = mid;
      else hi = mid - 1;
    }
    b = lo;
  }
  const int64_t r0 = int64_t(off[b]) + (tgt ? b : 0);
  const int64_t r1 = int64_t(off[b + 1]) + (tgt ? b : -1);
  cur->b = b;
  cur->r0 = r0;
  cur->r1 = r1;
  return (r >= r0 && r <= r1) ? b : -1;
}

// Repetition penalty: the request's penalized columns within a unit held in
// shared memory are set to -inf (they leave its top-k list; the kept-set
// kernel adds them back with the row's own values); those in the unit's
// ragged tail, read directly, are returned as lane bits to drop.
template <int DT>
__device__ __forceinline__ uint32_t mask_penalized(char* stage, const Desc& d, const RowSet& S,
                                                   int cps, int lane) {
  const int u = d.chunk / cps;
  const int64_t srow = int64_t(d.req) * (S.nch + 1);
  const int base = S.pbase[d.req];
  const int lo = S.pstart[srow + u], hi = S.pstart[srow + u + 1];
  const int c0 = d.chunk * kChunk;
  uint32_t drop = 0u;
  for (int i = lo + lane; i < hi; i += 32) {
    const int x = S.pen[base + i].col - c0;
    if (x >= 0 && x < d.n_smem) {
      if constexpr (DT == TT_F32) reinterpret_cast<float*>(stage)[x] = -INFINITY;
      else reinterpret_cast<uint16_t*>(stage)[x] = 0xff80u;  // bf16 -inf
    } else if (x >= d.n_smem && x < d.n) {
      drop |= 1u << (x - d.n_smem);
    }
  }
  drop = __reduce_or_sync(0xffffffffu, drop);
  __syncwarp();
  return drop;
}

template <int DT>
__device__ __forceinline__ float lane_elem(const uint4& v, int q) {
  if constexpr (DT == TT_F32) {
    return __uint_as_float(q == 0 ? v.x : q == 1 ? v.y : q == 2 ? v.z : v.w);
  } else {
    const int h = q >> 1;
    const uint32_t w = h == 0 ? v.x : h == 1 ? v.y : h == 2 ? v.z : v.w;
    return __uint_as_float((q & 1) ? (w & 0xffff0000u) : (w << 16));
  }
}

__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Largest raw logit of one lane's share of a whole chunk. The scale is
// positive and rounding is monotonic, so max(z * scale) = max(z) * scale
// exactly: the maximum is taken on the raw values (bf16 two at a time).
template <int DT>
__device__ __forceinline__ float raw_max_plain(const uint4* sv, int lane) {
  constexpr int VEC = DT == TT_F32 ? 4 : 8;
  constexpr int NV = kChunk / (VEC * 32);
  if constexpr (DT == TT_F32) {
    float m = -INFINITY;
#pragma unroll 4
    for (int v = 0; v < NV; ++v) {
      const uint4 w = sv[v * 32 + lane];
      m = fmaxf(m, fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                         fmaxf(__uint_as_float(w.z), __uint_as_float(w.w))));
    }
    return m;
  } else {
    uint32_t m2 = 0xff80ff80u;  // two bf16 -inf
#pragma unroll 4
    for (int v = 0; v < NV; ++v) {
      const uint4 w = sv[v * 32 + lane];
      m2 = max_bf16x2(m2, max_bf16x2(max_bf16x2(w.x, w.y), max_bf16x2(w.z, w.w)));
    }
    return fmaxf(__uint_as_float(m2 << 16), __uint_as_float(m2 & 0xffff0000u));
  }
}

// A unit's family as a consumer sees it: the kernel's arguments and which of
// the two families (d.set) the unit belongs to, so that both families share
// one copy of the code; the row's base is formed only where a ragged tail is
// read directly.
struct RowView {
  const RowPassArgs& a;
  float scale;
  __device__ __forceinline__ const char* row(const Desc& d) const {
    return d.set ? a.t.data + d.row * a.t.stride_bytes : a.d.data + d.row * a.d.stride_bytes;
  }
};

// One consumer warp reduces one chunk held in shared memory (plus a ragged
// tail of fewer than 16 bytes read directly) to (max, sum of 2^(s - max)).
// The stage is read twice (max, then sum) rather than held in registers.
template <int DT, bool PLAIN>
__device__ __forceinline__ void reduce_stage(const uint4* sv, const Desc& d, float scale,
                                             int lane, float& mx, float& sum) {
  constexpr int VEC = DT == TT_F32 ? 4 : 8;  // elements per 16 bytes
  constexpr int NV = kChunk / (VEC * 32);    // 16-byte vectors per lane
  if constexpr (PLAIN) {
    mx = fmaxf(mx, raw_max_plain<DT>(sv, lane) * scale);
  } else {
#pragma unroll 4
    for (int v = 0; v < NV; ++v) {
      const uint4 w = sv[v * 32 + lane];
#pragma unroll
      for (int q = 0; q < VEC; ++q) {
        const int e = (v * 32 + lane) * VEC + q;
        if (e < d.n_smem && e != d.excl) mx = fmaxf(mx, lane_elem<DT>(w, q) * scale);
      }
    }
  }
  if (mx == -INFINITY) return;
#pragma unroll 4
  for (int v = 0; v < NV; ++v) {
    const uint4 w = sv[v * 32 + lane];
#pragma unroll
    for (int q = 0; q < VEC; ++q) {
      const int e = (v * 32 + lane) * VEC + q;
      if (PLAIN || (e < d.n_smem && e != d.excl))
        sum += ex2_approx(fmaf(lane_elem<DT>(w, q), scale, -mx));
    }
  }
}

// The chunks that are not whole or hold the scored column -- at most two per
// row -- take this out-of-line copy, which keeps the consumer loop's code (and
// its share of the instruction cache) to the whole-chunk path.
template <int DT>
__device__ __noinline__ float2 reduce_stage_edge(const uint4* sv, int n_smem, int excl, float scale,
                                                 int lane, float mx) {
  Desc d;
  d.n_smem = n_smem;  // the only fields the per-element checks read
  d.excl = excl;
  float sum = 0.f;
  reduce_stage<DT, false>(sv, d, scale, lane, mx, sum);
  return make_float2(mx, sum);
}

template <int DT>
__device__ __forceinline__ void reduce_chunk(const char* stage, const Desc& d, const RowView& S,
                                             int lane, float& m_out, float& s_out) {
  const uint4* sv = reinterpret_cast<const uint4*>(stage);
  const float scale = S.scale;
  // ragged tail: at most 7 columns beyond the bulk copy, one per lane
  float ztail = -INFINITY;
  const int tail = d.n - d.n_smem;
  if (lane < tail) {
    const int e = d.n_smem + lane;
    if (e != d.excl) {
      ztail = load_logit<DT>(S.row(d), int64_t(d.chunk) * kChunk + e) * scale;
    }
  }
  float mx = ztail, sum = 0.f;
  if (d.n_smem == kChunk && d.excl < 0) {
    reduce_stage<DT, true>(sv, d, scale, lane, mx, sum);
  } else {
    const float2 r = reduce_stage_edge<DT>(sv, d.n_smem, d.excl, scale, lane, mx);
    mx = r.x;
    sum = r.y;
  }
  if (ztail != -INFINITY) sum += ex2_approx(ztail - mx);
  m_out = mx;
  s_out = sum;
}

// Candidate order of the top-k: larger logit first, then smaller column.
__device__ __forceinline__ bool cand_before(float v1, int c1, float v2, int c2) {
  return v1 > v2 || (v1 == v2 && c1 < c2);
}

// Largest logit of one 16-byte vector (4 fp32 or 8 bf16 logits).
template <int DT>
__device__ __forceinline__ float vec_max(const uint4& w) {
  if constexpr (DT == TT_F32) {
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                 fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
  } else {
    const uint32_t m = max_bf16x2(max_bf16x2(w.x, w.y), max_bf16x2(w.z, w.w));
    return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
  }
}

// Partial of one chunk of a nucleus row (all its columns, the scored one
// included) from a unit held in shared memory plus its ragged tail read
// directly: the chunk's largest z * scale and the sum of 2^(s - m), each
// 16-byte vector's terms added plainly and the vectors' sums in compensated
// pairs (TwoSum), so that the row's normaliser -- against which the top-p cut
// is placed -- stays within a few 1e-7 of exact.
template <int DT>
__device__ __forceinline__ Partial nuc_chunk_partial(const char* stage, const Desc& d,
                                                     const char* row, float scale, int c,
                                                     int lane) {
  constexpr int VEC = DT == TT_F32 ? 4 : 8;
  const int lo = c * kChunk;                       // first column of the chunk in the unit
  const int hi = min(d.n, lo + kChunk);            // its end
  const int smem_hi = min(hi, d.n_smem);           // columns held in shared memory
  const int col0 = d.chunk * kChunk;
  const uint4* sv = reinterpret_cast<const uint4*>(stage);
  const int v0 = lo / VEC, v1 = smem_hi / VEC;     // whole vectors (lo is a multiple of VEC)
  const int t = smem_hi + lane;                    // the ragged tail: one column per lane
  const float zt = (t < hi && t >= d.n_smem) ? load_logit<DT>(row, int64_t(col0) + t) : -INFINITY;
  float zmax = zt;
  for (int v = v0 + lane; v < v1; v += 32) zmax = fmaxf(zmax, vec_max<DT>(sv[v]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) zmax = fmaxf(zmax, __shfl_xor_sync(0xffffffffu, zmax, o));
  const float m = __fmul_rn(zmax, scale);
  float hs = 0.f, ls = 0.f;  // compensated sum (hi, lo)
  if (m > -INFINITY) {
    auto add = [&](float x) {
      const float sx = __fadd_rn(hs, x), bb = __fsub_rn(sx, hs);
      ls = __fadd_rn(ls, __fadd_rn(__fsub_rn(hs, __fsub_rn(sx, bb)), __fsub_rn(x, bb)));
      hs = sx;
    };
    for (int v = v0 + lane; v < v1; v += 32) {  // one vector's terms summed plainly
      const uint4 w = sv[v];
      float blk = 0.f;
#pragma unroll
      for (int q = 0; q < VEC; ++q) blk += ex2_approx(fmaf(lane_elem<DT>(w, q), scale, -m));
      add(blk);
    }
    if (zt > -INFINITY) add(ex2_approx(fmaf(zt, scale, -m)));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float oh = __shfl_xor_sync(0xffffffffu, hs, o), ol = __shfl_xor_sync(0xffffffffu, ls, o);
      ls = __fadd_rn(ls, ol);
      add(oh);
    }
  }
  return Partial{m, __fadd_rn(hs, ls)};
}

// One consumer warp writes the top-K (value, column) list of one unit held in
// shared memory (its whole 16-byte vectors) plus a ragged tail of fewer than
// 16 bytes read directly, ordered by cand_before, padded with (-inf, -1);
// columns are absolute. Each lane owns 16 vectors and keeps their maxima in
// registers. A threshold at or below the unit's K-th largest element bounds
// the candidates:
//   tau1, the K-th largest of the 64 values formed by each lane's two largest
//   vector maxima (two bitonic sorts and a merge; K <= 32); K vectors reach
//   it, so K elements do. Usually about K vectors reach tau1 and their
//   elements at or above it are the candidates.
//   When more than 32 vectors reach tau1 (large logits crowded into few
//   lanes), tau2, the K-th largest vector maximum, is found among them: by
//   counting when they are at most 64, else by a radix search over the maxima
//   in registers, and about K vectors reach it whatever the crowding.
// The candidates are gathered in `scratch` and ranked by counting; more than
// kCandCap (runs of equal logits) take K rounds of a warp-wide extraction over
// the same vectors instead. The work per unit is thus nearly the same for
// every unit, which keeps the stage ring from waiting on one slow warp.
template <int DT>
__device__ void select_unit(const char* stage, const Desc& d, const RowView& S, int lane, int K,
                            Cand* scratch, Cand* out, uint32_t tail_drop = 0u) {
  constexpr int VEC = DT == TT_F32 ? 4 : 8;  // logits per 16-byte vector
  constexpr int NV = kChunk * 4 / (16 * 32);   // vectors per lane in one stage
  constexpr uint32_t kTailBit = 1u << NV;      // flag of the lane's tail element
  const float kNaN = __int_as_float(0x7fffffff);
  const uint4* sv = reinterpret_cast<const uint4*>(stage);
  const int col0 = d.chunk * kChunk;
  const int nvec = d.n_smem / VEC;  // whole vectors delivered (the copy moves 16-byte units)
  // this lane's vectors v < nvl lie within the copy
  const int nvl = max(0, min(NV, (nvec - lane + 31) >> 5));
  const bool has_tail = lane < d.n - d.n_smem && !((tail_drop >> lane) & 1u);
  // the tail element, NaN where the lane has none (NaN never compares >=)
  float zt = kNaN;
  if (has_tail) {
    zt = load_logit<DT>(S.row(d), int64_t(col0) + d.n_smem + lane);
  }
  const uint32_t valid = ((1u << nvl) - 1) | (has_tail ? kTailBit : 0u);
  float vm[NV];  // vector maxima; -inf for a vector past the copy
  float m1 = has_tail ? zt : -INFINITY, m2 = -INFINITY;  // the lane's two largest
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const float x = vec_max<DT>(sv[v * 32 + lane]);
    vm[v] = v < nvl ? x : -INFINITY;
    m2 = fmaxf(m2, fminf(m1, vm[v]));
    m1 = fmaxf(m1, vm[v]);
  }
  auto at_or_above = [&](float t) {
    uint32_t f = zt >= t ? kTailBit : 0u;
#pragma unroll
    for (int v = 0; v < NV; ++v) f |= vm[v] >= t ? (1u << v) : 0u;
    return f & valid;
  };
  // the 32 largest of the 64: half-cleaner of (m1 descending, m2 ascending)
  const float top = warp_merge_desc(fmaxf(warp_sort<true>(m1, lane), warp_sort<false>(m2, lane)),
                                    lane);
  float tau = __shfl_sync(0xffffffffu, top, K - 1);
  uint32_t flags = at_or_above(tau);
  const int nf = __popc(flags);
  const int F1 = int(__reduce_add_sync(0xffffffffu, unsigned(nf)));
  if (F1 > kDirectCap) {
    // tau2: the K-th largest maximum; every vector that reaches it reaches tau1
    if (F1 <= kLevel2Cap) {
      int incl = nf;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
      }
      float* vals = reinterpret_cast<float*>(scratch);
      int p = incl - nf;
#pragma unroll
      for (int v = 0; v < NV; ++v)
        if (flags & (1u << v)) vals[p++] = vm[v];
      if (flags & kTailBit) vals[p] = zt;
      __syncwarp();
      // the K-th largest w is the largest with #{values >= w} >= K; lane l
      // tests values l and l + 32 (NaN: absent)
      const float w0 = lane < F1 ? vals[lane] : kNaN;
      const float w1 = lane + 32 < F1 ? vals[lane + 32] : kNaN;
      int c0 = 0, c1 = 0;
#pragma unroll 4
      for (int j = 0; j < F1; ++j) {
        const float x = vals[j];
        c0 += x >= w0;
        c1 += x >= w1;
      }
      float best = -INFINITY;
      if (c0 >= K) best = w0;
      if (c1 >= K) best = fmaxf(best, w1);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, o));
      tau = best;
      __syncwarp();  // the values are read before the scratch takes candidates
    } else {
      // radix search on order-preserving keys (x >= 0: bits | 2^31, else
      // ~bits): the largest key t with #{maxima whose key >= t} >= K, one bit
      // at a time. A probe's float is compared, so probes below the key of
      // -inf (NaN floats) never pass: a K-th largest of -inf ends at t = 0.
      uint32_t t = 0;
      for (int b = 31; b >= 0; --b) {
        const uint32_t probe = t | (1u << b);
        const float pf = __uint_as_float((probe & 0x80000000u) ? (probe & 0x7fffffffu) : ~probe);
        int c = zt >= pf;
#pragma unroll
        for (int v = 0; v < NV; ++v) c += vm[v] >= pf;
        if (int(__reduce_add_sync(0xffffffffu, unsigned(c))) >= K) t = probe;
      }
      tau = t < 0x007fffffu ? -INFINITY
                            : __uint_as_float((t & 0x80000000u) ? (t & 0x7fffffffu) : ~t);
    }
    flags = at_or_above(tau);
  }
  const float tau2 = tau;

  // candidates: the elements at or above tau2, counted, then written at their
  // lane's offset in the warp
  int nc = (flags & kTailBit) ? 1 : 0;
  for (uint32_t f = flags & (kTailBit - 1); f; f &= f - 1) {
    const uint4 w = sv[(__ffs(f) - 1) * 32 + lane];
#pragma unroll
    for (int q = 0; q < VEC; ++q) nc += lane_elem<DT>(w, q) >= tau2;
  }
  int cincl = nc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, cincl, o);
    if (lane >= o) cincl += x;
  }
  const int C = __shfl_sync(0xffffffffu, cincl, 31);
  if (C <= kCandCap) {
    int p = cincl - nc;
    if (flags & kTailBit) scratch[p++] = Cand{zt, d.n_smem + lane};
    for (uint32_t f = flags & (kTailBit - 1); f; f &= f - 1) {
      const int v = __ffs(f) - 1;
      const uint4 w = sv[v * 32 + lane];
#pragma unroll
      for (int q = 0; q < VEC; ++q) {
        const float x = lane_elem<DT>(w, q);
        if (x >= tau2) scratch[p++] = Cand{x, (v * 32 + lane) * VEC + q};
      }
    }
    __syncwarp();
    for (int i = lane; i < C; i += 32) {
      const Cand ci = scratch[i];
      int r = 0;
#pragma unroll 4
      for (int j = 0; j < C; ++j) {
        const Cand cj = scratch[j];
        r += cand_before(cj.v, cj.c, ci.v, ci.c);
      }
      if (r < K) out[r] = Cand{ci.v, col0 + ci.c};
    }
    for (int r = C + lane; r < K; r += 32) out[r] = Cand{-INFINITY, -1};
  } else {
    // exact extraction over the flagged vectors: round r takes the best
    // element after round r-1's pick
    float pv = INFINITY;
    int pc = -1;
    for (int r = 0; r < K; ++r) {
      float bv = -INFINITY;
      int bc = 0x7fffffff;
      bool f = false;
      auto consider = [&](float x, int c) {
        if (cand_before(pv, pc, x, c) && (!f || cand_before(x, c, bv, bc))) {
          bv = x;
          bc = c;
          f = true;
        }
      };
      if (flags & kTailBit) consider(zt, d.n_smem + lane);
      for (uint32_t g = flags & (kTailBit - 1); g; g &= g - 1) {
        const int v = __ffs(g) - 1;
        const uint4 w = sv[v * 32 + lane];
#pragma unroll
        for (int q = 0; q < VEC; ++q) consider(lane_elem<DT>(w, q), (v * 32 + lane) * VEC + q);
      }
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
      if (lane == 0) out[r] = f ? Cand{bv, col0 + bc} : Cand{-INFINITY, -1};
      if (f) {
        pv = bv;
        pc = bc;
      } else {
        pv = -INFINITY;  // nothing left: pad the rest
        pc = 0x7fffffff;
      }
    }
  }
  __syncwarp();  // the scratch is free for the next unit
}

template <int DTD, int DTT, int SEL>
__global__ void __launch_bounds__(kThreads, 3) rowpass_kernel(RowPassArgs a) {
  using R = Ring<DTD, DTT, SEL>;
  extern __shared__ __align__(128) char smem[];
  char* stages = smem;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kRingBytes);
  uint64_t* empty = full + R::kStages;
  Desc* desc = reinterpret_cast<Desc*>(empty + R::kStages);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // a consumer warp's candidate scratch (filtered rows only)
  Cand* scratch = reinterpret_cast<Cand*>(desc + R::kStages) + (SEL ? warp * kCandCap : 0);

  if (threadIdx.x == 0) {
    for (int s = 0; s < R::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const int64_t G = gridDim.x, g = blockIdx.x;
      // units (stages) per row and in all of each family
      const int upr_t = (a.t.nch + R::kCpsT - 1) / R::kCpsT;
      const int upr_d = (a.d.nch + R::kCpsD - 1) / R::kCpsD;
      const int64_t items_t = a.rows_t * upr_t, items_d = a.rows_d * upr_d;
      bool ok = true;
      int it = 0;
      int64_t cached_row = -1, cached_drow = -1;
      int cached_excl = -1;
      __shared__ ExclCursor cursor;
      __shared__ ReqCursor rcur_d, rcur_t;
      cursor.b = -1;
      rcur_d.b = rcur_t.b = -1;
      bool cached_need = true;
      // Queues chunk `chunk` of row `row` (tgt: a target row, else a draft
      // row) on the next stage; false once a wait has run out.
      bool late = false;  // past the grid-dependency wait
      auto issue = [&](bool tgt, int64_t row, int unit) -> bool {
        Desc d;
        const RowSet* S;
        int esz, cps;
        d.row = row;
        if (tgt) {
          S = &a.t;
          esz = DTT == TT_F32 ? 4 : 2;
          cps = R::kCpsT;
          d.set = 1;
          if (row != cached_row) {
            cached_row = row;
            cached_excl = a.excl                ? a.excl[row]
                          : (late && a.excl_late) ? a.excl_late[row]
                                                  : excl_lookup(a, &cursor, row);
          }
          const int ex = cached_excl - unit * cps * kChunk;
          d.excl = (cached_excl >= 0 && ex >= 0 && ex < cps * kChunk) ? ex : -1;
        } else {
          S = &a.d;
          esz = DTD == TT_F32 ? 4 : 2;
          cps = R::kCpsD;
          d.set = 0;
          d.excl = -1;
          if (row != cached_drow) {
            cached_drow = row;
            cached_need = !a.d.need || a.d.need[row] != 0;
          }
          if (!cached_need) return true;  // no target position maps to this row
        }
        // (penalized families have top-k lists: the list-selecting variant only)
        d.req = (SEL == 2 && S->pen) ? req_lookup(tgt ? a.target_off : a.draft_off, a.B, tgt,
                                                  tgt ? &rcur_t : &rcur_d, row)
                                     : -1;
        d.chunk = unit * cps;
        const int c0 = d.chunk * kChunk;
        d.n = min(cps * kChunk, S->V - c0);
        const uint32_t bytes = uint32_t(d.n * esz) & ~15u;  // bulk copies move 16-byte units
        d.n_smem = int(bytes) / esz;
        const int s = it % R::kStages;
        const uint32_t par = ((it / R::kStages) & 1) ^ 1;
        if (!mbar_wait(&empty[s], par, a.wait_ns)) {
          report_error(a.err, a.epoch, TT_REQ_TIMEOUT);
          return false;
        }
        // every bulk copy is checked against the tensor before it is issued
        const char* src = S->data + d.row * S->stride_bytes + size_t(c0) * esz;
        const bool copy_ok = d.row >= 0 && d.row < S->n_rows && c0 >= 0 && d.n > 0 &&
                             (reinterpret_cast<uintptr_t>(src) & 15) == 0 &&
                             bytes <= uint32_t(R::kStageBytes);
        if (!copy_ok) {
          report_error(a.err, a.epoch, TT_REQ_INTERNAL);
          d.n = 0;
          d.n_smem = 0;
        }
        desc[s] = d;
        if (copy_ok && bytes > 0) {
          mbar_arrive_expect_tx(&full[s], bytes);
          bulk_copy_g2s(stages + size_t(s) * R::kStageBytes, src, bytes, &full[s]);
        } else {
          mbar_arrive(&full[s]);
        }
        ++it;
        return true;
      };
      // Queues items [i0, i1) of a family (item = row * units per row + unit),
      // walking rows and units without a division per item.
      auto walk = [&](bool tgt, int64_t i0, int64_t i1) {
        if (i0 >= i1) return;
        const int upr = tgt ? upr_t : upr_d;
        int64_t row = i0 / upr;
        int unit = int(i0 - row * upr);
        for (int64_t i = i0; ok && i < i1; ++i) {
          ok = issue(tgt, row, unit);
          if (++unit == upr) {
            unit = 0;
            ++row;
          }
        }
      };

      if (!a.work) {
        // fixed shares only: a block of target items, then a block of draft items
        const int64_t t_lo = items_t * g / G, t_hi = items_t * (g + 1) / G;
        const int64_t d_lo = items_d * g / G, d_hi = items_d * (g + 1) / G;
        walk(true, t_lo, t_hi);
        grid_dependency_wait();  // draft rows need the alignment's flags
        // the next grid may start now (the alignment grid is complete): its CTAs
        // are small enough to sit beside these and wait there for this grid's end
        grid_launch_dependents();
        walk(false, d_lo, d_hi);
      } else {
        // A fixed block of a.pre_eighths / 8 of the target items, streamed
        // while the alignment may still run (target rows do not depend on
        // it); then batches of the rest (target items, then draft items) from
        // the work counter, so that CTAs that started late or drew less
        // bandwidth take fewer and all finish together.
        const int64_t per = items_t * a.pre_eighths / 8 / G;
        walk(true, g * per, (g + 1) * per);
        grid_dependency_wait();  // the counters, flags and scored columns are ready
        late = true;
        grid_launch_dependents();  // as above
        const int64_t t_rest = G * per, n_rest_t = items_t - t_rest;
        const int64_t pool = n_rest_t + items_d;
        // Guided self-scheduling over kWorkShards sub-pools: CTA g starts on
        // shard g mod kWorkShards; a draw takes 1/(4 * its CTAs) of what is
        // left there (within [kGrabMin, kGrabMax] items), so draws are larger
        // early and small only at the end. A CTA whose shard runs dry moves
        // on to the next one. The next draw is made while the current batch
        // is queued, so the counter's round trip never stalls the ring.
        const int64_t ctas = max(int64_t(1), G / kWorkShards);
        auto draw_size = [&](int64_t left) -> int64_t {
          return max(int64_t(R::kGrabMin), min(int64_t(R::kGrabMax), left / (4 * ctas)));
        };
        for (int v = 0; ok && v < kWorkShards; ++v) {
          const int sh = int((g + v) % kWorkShards);
          const int64_t lo = pool * sh / kWorkShards, n = pool * (sh + 1) / kWorkShards - lo;
          unsigned long long* ctr = a.work + sh * kWorkStride;
          int64_t size = v == 0 ? draw_size(n / 2) : int64_t(R::kGrabMin);
          int64_t base = int64_t(atomicAdd(ctr, (unsigned long long)size));
          while (ok && base < n) {
            const int64_t size_next = draw_size(n - base - size);
            const int64_t next = int64_t(atomicAdd(ctr, (unsigned long long)size_next));
            const int64_t x0 = lo + base, x1 = lo + min(n, base + size);
            walk(true, t_rest + x0, t_rest + min(x1, n_rest_t));  // pool: target items first
            walk(false, max(x0, n_rest_t) - n_rest_t, x1 - n_rest_t);
            base = next;
            size = size_next;
          }
        }
      }
      // one end marker per consumer warp
      for (int w = 0; ok && w < kConsumerWarps; ++w) {
        const int s = it % R::kStages;
        const uint32_t par = ((it / R::kStages) & 1) ^ 1;
        if (!mbar_wait(&empty[s], par, a.wait_ns)) {
          report_error(a.err, a.epoch, TT_REQ_TIMEOUT);
          ok = false;
          break;
        }
        desc[s].row = -1;
        mbar_arrive(&full[s]);
        ++it;
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  // (one thread's launch_dependents counts for its whole CTA: only the
  // producer lane gives it, after its grid-dependency wait, because the next
  // grid reads the alignment's outputs before its own wait)
  for (int it = warp;; it += kConsumerWarps) {
    const int s = it % R::kStages;
    const uint32_t par = (it / R::kStages) & 1;
    if (!mbar_wait(&full[s], par, a.wait_ns)) {
      if (lane == 0) report_error(a.err, a.epoch, TT_REQ_TIMEOUT);
      break;
    }
    const Desc d = desc[s];
    if (d.row < 0) break;
    const char* stage = stages + size_t(s) * R::kStageBytes;
    const int cps = d.set ? R::kCpsT : R::kCpsD;
    const int esz = (d.set ? DTT : DTD) == TT_F32 ? 4 : 2;
    if constexpr (SEL == 2) {
      const RowSet& S = d.set ? a.t : a.d;
      if (S.nucleus) {  // nucleus rows: the compensated partials of all the unit's columns
        const RowView V = {a, S.scale};
#pragma unroll 1
        for (int c = 0; c < cps && c * kChunk < d.n; ++c) {
          const Partial pc =
              (d.set ? DTT : DTD) == TT_F32
                  ? nuc_chunk_partial<TT_F32>(stage, d, V.row(d), S.scale, c, lane)
                  : nuc_chunk_partial<TT_BF16>(stage, d, V.row(d), S.scale, c, lane);
          if (lane == 0) S.part[d.row * S.nch + d.chunk + c] = pc;
        }
        __syncwarp();
        if (lane == 0 && !(blockIdx.x == 0 && it == a.stall_stage))
          mbar_arrive(&empty[s]);  // the stage's bytes are consumed
        continue;
      }
    }
    if (SEL && (d.set ? a.t : a.d).top_k > 0) {  // filtered rows: the unit's top-k list
      const RowSet& S = d.set ? a.t : a.d;
      Cand* out = S.cand + (d.row * S.nlist + d.chunk / cps) * cand_stride(S.top_k);
      const RowView V = {a, S.scale};
      uint32_t drop = 0u;
      if constexpr (SEL == 2) {
        if (S.pen && d.req >= 0) {
          char* wstage = stages + size_t(s) * R::kStageBytes;
          drop = (d.set ? DTT : DTD) == TT_F32 ? mask_penalized<TT_F32>(wstage, d, S, cps, lane)
                                               : mask_penalized<TT_BF16>(wstage, d, S, cps, lane);
        }
      }
      if constexpr (DTD == DTT) {
        select_unit<DTT>(stage, d, V, lane, S.top_k, scratch, out, drop);
      } else if (d.set) {
        select_unit<DTT>(stage, d, V, lane, S.top_k, scratch, out, drop);
      } else {
        select_unit<DTD>(stage, d, V, lane, S.top_k, scratch, out, drop);
      }
      if (lane == 0 && !(blockIdx.x == 0 && it == a.stall_stage))
        mbar_arrive(&empty[s]);  // the stage's bytes are consumed
      continue;
    }
    // the unit's chunks (two for bf16 rows), each reduced on its own by one
    // copy of the code; the results are named, not indexed, to stay in registers
    float m0 = -INFINITY, s0 = 0.f, m1 = -INFINITY, s1 = 0.f;
#pragma unroll 1
    for (int c = 0; c < cps; ++c) {
      const int lo = c * kChunk;
      if (lo >= d.n) break;
      Desc e = d;
      e.chunk = d.chunk + c;
      e.n = min(kChunk, d.n - lo);
      e.n_smem = max(0, min(kChunk, d.n_smem - lo));
      e.excl = (d.excl >= lo && d.excl < lo + kChunk) ? d.excl - lo : -1;
      float mc = -INFINITY, sc = 0.f;
      // fp32 rows: one copy for both families; bf16 rows: one per family (shared,
      // the kernel needs more registers than the decision kernel beside it leaves)
      if constexpr (DTD == TT_F32 && DTT == TT_F32) {
        reduce_chunk<TT_F32>(stage + size_t(lo) * esz, e,
                             RowView{a, d.set ? a.t.scale : a.d.scale}, lane, mc, sc);
      } else if (d.set) {
        reduce_chunk<DTT>(stage + size_t(lo) * esz, e, RowView{a, a.t.scale}, lane, mc, sc);
      } else {
        reduce_chunk<DTD>(stage + size_t(lo) * esz, e, RowView{a, a.d.scale}, lane, mc, sc);
      }
      if (c == 0) {
        m0 = mc;
        s0 = sc;
      } else {
        m1 = mc;
        s1 = sc;
      }
    }
    __syncwarp();
    // (test hook: in CTA 0 the consumer of its stall_stage-th stage never frees
    // it, so the producer's bounded wait for it runs out, then the others')
    if (lane == 0 && !(blockIdx.x == 0 && it == a.stall_stage))
      mbar_arrive(&empty[s]);  // the stage's bytes are consumed
    const RowSet& S = d.set ? a.t : a.d;
    if (d.n <= 0) continue;  // nothing copied (a failed check: the row may not exist)
    warp_merge_ms(m0, s0);
    if (lane == 0) S.part[d.row * S.nch + d.chunk] = Partial{m0, s0};
    if (cps > 1 && kChunk < d.n) {
      warp_merge_ms(m1, s1);
      if (lane == 0) S.part[d.row * S.nch + d.chunk + 1] = Partial{m1, s1};
    }
  }
}

template <int DTD, int DTT, int SEL>
int& resident_per_sm() {
  static int per_sm = 0;
  return per_sm;
}

template <int DTD, int DTT, int SEL>
cudaError_t preload_t() {
  using R = Ring<DTD, DTT, SEL>;
  cudaError_t e = cudaFuncSetAttribute(rowpass_kernel<DTD, DTT, SEL>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(R::kSmem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(rowpass_kernel<DTD, DTT, SEL>,
                           cudaFuncAttributePreferredSharedMemoryCarveout,
                           int(cudaSharedmemCarveoutMaxShared));
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rowpass_kernel<DTD, DTT, SEL>,
                                                    kThreads, R::kSmem);
  if (e != cudaSuccess) return e;
  resident_per_sm<DTD, DTT, SEL>() = per_sm < 1 ? 1 : per_sm;
  return cudaSuccess;
}

template <int DTD, int DTT, int SEL>
cudaError_t launch_rowpass_t(const RowPassArgs& a, cudaStream_t stream, int sm_count, bool pdl) {
  using R = Ring<DTD, DTT, SEL>;
  const int per_sm = resident_per_sm<DTD, DTT, SEL>();
  if (per_sm == 0) return cudaErrorNotReady;  // preload_rowpass() was not called
  const int64_t total = a.rows_t * ((a.t.nch + R::kCpsT - 1) / R::kCpsT) +
                        a.rows_d * ((a.d.nch + R::kCpsD - 1) / R::kCpsD);
  if (total == 0) return cudaSuccess;
  const int64_t grid = std::min<int64_t>(total, int64_t(sm_count) * per_sm);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = R::kSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, rowpass_kernel<DTD, DTT, SEL>, a);
}

template <int DTD, int DTT>
cudaError_t preload_pair() {
  cudaError_t e = preload_t<DTD, DTT, 0>();
  if (e == cudaSuccess) e = preload_t<DTD, DTT, 1>();
  return e != cudaSuccess ? e : preload_t<DTD, DTT, 2>();
}

// Variants: 0 partials only; 1 top-k lists for filtered families; 2 lists with
// the repetition penalty's masking and the nucleus rows' partials (kept apart
// so that plain filtered rows run the smaller consumer loop).
template <int DTD, int DTT>
cudaError_t launch_pair(const RowPassArgs& a, cudaStream_t stream, int sm_count, bool pdl) {
  if (a.d.pen || a.t.pen || a.d.nucleus || a.t.nucleus)
    return launch_rowpass_t<DTD, DTT, 2>(a, stream, sm_count, pdl);
  if (a.d.top_k > 0 || a.t.top_k > 0) return launch_rowpass_t<DTD, DTT, 1>(a, stream, sm_count, pdl);
  return launch_rowpass_t<DTD, DTT, 0>(a, stream, sm_count, pdl);
}

}  // namespace

cudaError_t preload_rowpass() {
  cudaError_t e;
  if ((e = preload_pair<TT_F32, TT_F32>()) != cudaSuccess) return e;
  if ((e = preload_pair<TT_F32, TT_BF16>()) != cudaSuccess) return e;
  if ((e = preload_pair<TT_BF16, TT_F32>()) != cudaSuccess) return e;
  return preload_pair<TT_BF16, TT_BF16>();
}

namespace {

// Test hook of the bounded waits, read from the environment once per process
// (off unless set): TT_TEST_STALL_STAGE=n makes CTA 0 of the first
// TT_TEST_STALL_LAUNCHES row-pass launches (default 1) hold the stage of its
// n-th consumer step, with every pipeline wait of those launches limited to
// TT_TEST_WAIT_MS milliseconds, so that a test can watch the waits run out and
// the call report TT_REQ_TIMEOUT, then see the next launches run normally.
struct StallHook {
  int stall_stage = -1;
  uint64_t wait_ns = kWaitLimitNs;
  std::atomic<int> launches_left{0};
  StallHook() {
    if (const char* v = std::getenv("TT_TEST_STALL_STAGE")) stall_stage = std::atoi(v);
    if (stall_stage < 0) return;
    if (const char* v = std::getenv("TT_TEST_WAIT_MS")) {
      const long long ms = std::atoll(v);
      if (ms > 0) wait_ns = uint64_t(ms) * 1000000ull;
    }
    int n = 1;
    if (const char* v = std::getenv("TT_TEST_STALL_LAUNCHES")) n = std::atoi(v);
    launches_left.store(n > 0 ? n : 0);
  }
};

StallHook& stall_hook() {
  static StallHook hook;  // initialised once, thread-safe
  return hook;
}

}  // namespace

cudaError_t launch_rowpass(const RowPassArgs& args, int dt_d, int dt_t, cudaStream_t stream,
                           int sm_count, bool pdl) {
  RowPassArgs a = args;
  a.stall_stage = -1;
  a.wait_ns = kWaitLimitNs;
  StallHook& hook = stall_hook();
  if (hook.stall_stage >= 0 && hook.launches_left.fetch_sub(1) > 0) {
    a.stall_stage = hook.stall_stage;
    a.wait_ns = hook.wait_ns;
  }
  if (dt_d == TT_F32 && dt_t == TT_F32) return launch_pair<TT_F32, TT_F32>(a, stream, sm_count, pdl);
  if (dt_d == TT_F32 && dt_t == TT_BF16) return launch_pair<TT_F32, TT_BF16>(a, stream, sm_count, pdl);
  if (dt_d == TT_BF16 && dt_t == TT_F32) return launch_pair<TT_BF16, TT_F32>(a, stream, sm_count, pdl);
  return launch_pair<TT_BF16, TT_BF16>(a, stream, sm_count, pdl);
}

}  // namespace tt
