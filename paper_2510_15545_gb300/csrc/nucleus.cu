// nucleus.cu -- verification under top-p without top-k (the nucleus rows of the
// paper's generation hyperparameters, App. F: T = 0.6 with top-p 0.9 or 0.95
// for the Llama-3.1-70B and DeepSeek-R1-Distill targets).
//
// A nucleus row keeps the shortest prefix of its columns, in the order larger
// logit first and then smaller column, whose probability mass at temperature T
// reaches top_p: every column whose mass before it is below top_p. The kept set
// can span thousands of columns, so it is not held as a list: it is the columns
// ranked at or before the last kept one (tau, tau_col), with kept probability
// 2^(z * scale - M) / S and its mass per 2048-column chunk.
//
// nucleus_kernel finds it exactly, one CTA per row, from the row's logits and
// the row pass's compensated partials of all its columns (which give the row
// maximum M and the row's total):
//  0. usually in one pass over the row: every column within kCandDelta = 14
//     log2 units of M is gathered in shared memory (on the paper's settings
//     the cut lies within about 13 units), the candidates' fixed-point masses
//     are binned as in step 1, and the crossing bucket is walked as in step 3
//     (one lane per candidate when it holds at most 32). Rows whose candidates
//     overflow the buffer or do not reach the cut take steps 1-4:
//  1. a histogram of delta = M - z * scale in buckets of 1/32 (log2 units) over
//     [0, 40), with counts and masses 2^-delta in 40-bit fixed point, so that
//     sums are exact in any order (columns at delta >= 40 weigh less than
//     2^-40 of the maximum and are not counted);
//  2. the bucket where the running mass, largest logits first, reaches top_p
//     of the total: every column of an earlier bucket is kept, none of a later
//     one; a crossing bucket of more than kRefine columns is split again by a
//     finer histogram of its range (twice at most: the last level holds one
//     fp32 value of delta per bucket);
//  3. the crossing bucket's columns are gathered in shared memory, and walked
//     by logit value from the largest: each value's run of tied columns (equal
//     mass) either lies wholly before the cut or holds it, and then the number
//     of its columns kept follows from the run's mass, the smallest columns of
//     the run first;
//  4. the chunk masses of the kept columns (the gathering pass adds those of
//     the earlier buckets), their total S and the header.
// decide_nucleus_kernel is the decision over nucleus target rows: p(t_j) and
// the accept test as elsewhere, and the residual (or bonus) draw at two
// levels, the chunk from the kept chunk masses and the column from that chunk
// re-read, in column order.
#include <algorithm>
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"
#include "tt_f2.cuh"

namespace tt {

namespace {

constexpr int kNT = 256;               // threads of the nucleus kernels
constexpr int kNW = kNT / 32;
constexpr int kBuckets = 1280;         // histogram buckets per level
constexpr float kDeltaMax = 40.f;      // level-0 range of delta (log2 units)
constexpr float kBucketsPerUnit = 32.f;  // level-0 buckets per log2 unit
constexpr int kLevels = 3;             // the level-0 histogram and two refinements
constexpr int kRefine = 256;           // a crossing bucket with more columns is split again
constexpr int kGather = 4096;          // columns held in shared memory (candidates, crossing bucket)
constexpr float kCandDelta = 14.f;     // candidates: delta below this (log2 units)
constexpr int kCross = 256;            // candidates of the crossing bucket held apart
constexpr int kRegion = kGather / kNW;  // candidates per warp's region of the buffer
constexpr int kUnitBins = 16;          // candidate counts per whole log2 unit of delta
constexpr int kRetryCands = 3200;      // candidates a second pass may take (of kGather)
constexpr float kMinBar = 8.f;         // lowest bar of a second pass
// Rows of at most kWarpRowMax columns: one warp per row (nucleus_warp_kernel),
// candidates within kWCandDelta log2 units of the maximum, at most kWCap.
constexpr int kWarpRowMax = 8192;
constexpr float kWCandDelta = 12.f;
constexpr int kWCap = 512;
constexpr int kWBuckets = int(kWCandDelta) * 32 + 32;
constexpr int kWWarps = 8;
constexpr int kWChunks = kWarpRowMax / kChunk;
// buckets of the candidates' delta (a little past kCandDelta: the fp32 delta of
// a candidate may round up to it)
constexpr int kCandBuckets = int(kCandDelta) * 32 + 32;
constexpr float kFix = 1099511627776.f;  // 2^40: fixed-point scale of the masses

__device__ __forceinline__ float load_dt(const char* row, int dt, int64_t col) {
  return dt == TT_F32 ? load_logit<TT_F32>(row, col) : load_logit<TT_BF16>(row, col);
}

// The bucket path of delta: level 0 (1/32 of a log2 unit), then each of the
// kBuckets parts of the level above; -1 at level 0 for delta >= kDeltaMax.
struct Path {
  int b[kLevels];
};

__device__ __forceinline__ Path bucket_path(float delta) {
  Path p;
  const float f0 = delta * kBucketsPerUnit;  // exact (a power of two)
  p.b[0] = (f0 >= 0.f && delta < kDeltaMax) ? int(f0) : -1;
  const float r0 = delta - float(p.b[0]) * (1.f / kBucketsPerUnit);  // exact
  const float f1 = r0 * (kBucketsPerUnit * kBuckets);
  p.b[1] = min(kBuckets - 1, max(0, int(f1)));
  const float f2 = (f1 - float(p.b[1])) * float(kBuckets);
  p.b[2] = min(kBuckets - 1, max(0, int(f2)));
  return p;
}

// -1: the path lies before (larger logits than) the crossing path's bucket at
// the given level, 0: inside it, 1: after it. Levels above `level` are taken
// as equal to cross's (callers test those first).
__device__ __forceinline__ int path_cmp(const Path& p, const Path& cross, int level) {
  for (int l = 0; l <= level; ++l) {
    if (p.b[l] < cross.b[l]) return -1;
    if (p.b[l] > cross.b[l]) return 1;
  }
  return 0;
}


// Shared memory of one nucleus CTA (about 58 KB: three CTAs fit on an SM).
struct NucSmem {
  unsigned int cnt[kBuckets];
  unsigned long long mass[kBuckets];
  unsigned long long cacc[kMaxChunksPerRow];  // kept mass per chunk
  Cand gz[kGather];                           // gathered columns (z, column)
  Cand gc[kCross];                            // candidates of the crossing bucket
  unsigned long long wsum[kNW];
  unsigned long long wmax[kNW];
  F2 wf2[kNW];
  int wcnt[kNW];
  int n_gz;
  int n_gc;
  int wn[kNW];  // candidates per warp region
  float ucnt[kUnitBins];  // estimated candidates per whole log2 unit of delta
  int todo[kNT];  // rows of the current tile left to this kernel
  int n_todo;
  float tau_v;  // the last kept column, found by one warp
  int tau_c;
  int cross;  // crossing bucket of the current level (-1: no bucket reaches the cut)
  unsigned long long before;  // mass of the columns ranked before the current range
};

// Block-wide sum of one 64-bit value per thread.
__device__ __forceinline__ unsigned long long block_sum_u64(unsigned long long v, NucSmem& s,
                                                            int lane, int warp) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) s.wsum[warp] = v;
  __syncthreads();
  unsigned long long t = 0;
#pragma unroll
  for (int w = 0; w < kNW; ++w) t += s.wsum[w];
  return t;
}

// Block-wide compensated sum of one pair per thread (the same on every thread).
__device__ __forceinline__ F2 block_sum_f2(F2 v, NucSmem& s, int lane, int warp) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    v = f2_add(v, F2{__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)});
  __syncthreads();
  if (lane == 0) s.wf2[warp] = v;
  __syncthreads();
  F2 t = {0.f, 0.f};
#pragma unroll
  for (int w = 0; w < kNW; ++w) t = f2_add(t, s.wf2[w]);
  return t;
}

// Block-wide (largest value below `below`, how many columns hold it) over
// n gathered columns.
__device__ __forceinline__ void block_max_count(const Cand* arr, NucSmem& s, int n, float below,
                                                int tid, float& vmax, int& count) {
  const int lane = tid & 31, warp = tid >> 5;
  float v = -INFINITY;
  for (int i = tid; i < n; i += kNT) {
    const float z = arr[i].v;
    if (z < below) v = fmaxf(v, z);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if (lane == 0) s.wmax[warp] = __float_as_uint(v) ^ (v < 0.f ? 0xffffffffu : 0x80000000u);
  __syncthreads();
  unsigned long long best = 0;
#pragma unroll
  for (int w = 0; w < kNW; ++w) best = max(best, s.wmax[w]);
  const uint32_t key = uint32_t(best);
  vmax = __uint_as_float(key & 0x80000000u ? key ^ 0x80000000u : ~key);
  int c = 0;
  for (int i = tid; i < n; i += kNT) c += arr[i].v == vmax;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __syncthreads();
  if (lane == 0) s.wcnt[warp] = c;
  __syncthreads();
  count = 0;
#pragma unroll
  for (int w = 0; w < kNW; ++w) count += s.wcnt[w];
}

__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Largest logit of a 16-byte vector (4 fp32 or 8 bf16 logits).
__device__ __forceinline__ float vector_max(const uint4& w, int dt) {
  if (dt == TT_F32)
    return fmaxf(fmaxf(__uint_as_float(w.x), __uint_as_float(w.y)),
                 fmaxf(__uint_as_float(w.z), __uint_as_float(w.w)));
  const uint32_t m = max_bf16x2(max_bf16x2(w.x, w.y), max_bf16x2(w.z, w.w));
  return fmaxf(__uint_as_float(m << 16), __uint_as_float(m & 0xffff0000u));
}

// One pass over a row's nvec whole 16-byte vectors by NTHR threads (this one
// is t), U loads in flight per thread: hit(v, w) for every vector w (the
// row's v-th) holding a logit above zc, found from the vector's maximum in a
// few instructions.
template <int NTHR, int U, class Hit>
__device__ __forceinline__ void scan_row(const uint4* rv, int nvec, int dt, float zc, int t,
                                         Hit&& hit) {
  for (int v0 = t; v0 < nvec; v0 += NTHR * U) {
    uint4 w[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = v0 + u * NTHR;
      if (v < nvec) w[u] = ld_stream_v4(rv + v);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = v0 + u * NTHR;
      if (v < nvec && vector_max(w[u], dt) > zc) hit(v, w[u]);
    }
  }
}

// The logits above zc of vector w (the row's v-th), passed to take(z, column).
template <class Take>
__device__ __forceinline__ void vector_candidates(const uint4& w, int dt, int v, float zc,
                                                  Take&& take) {
  const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
  if (dt == TT_F32) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float z = __uint_as_float(ww[q]);
      if (z > zc) take(z, v * 4 + q);
    }
  } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float z0 = __uint_as_float(ww[q] << 16), z1 = __uint_as_float(ww[q] & 0xffff0000u);
      if (z0 > zc) take(z0, v * 8 + 2 * q);
      if (z1 > zc) take(z1, v * 8 + 2 * q + 1);
    }
  }
}

// The cut among n gathered columns that hold it, `before` being the mass
// ranked before all of them: runs of equal logits from the largest; a run holds
// the cut or lies wholly before it, and the number of its columns kept follows
// from the run's mass (k columns kept while before + k' * mv < thr for
// k' < k), the smallest columns of the run first. Every thread calls; the last
// kept column is (tau, tau_col) on every thread.
__device__ void walk_runs(const Cand* arr, int n, unsigned long long before, double thr,
                          NucSmem& sm, float M, float scale, float& tau, int& tau_col) {
  const int tid = threadIdx.x;
  float below = INFINITY;
  for (int guard = 0; guard < n; ++guard) {
    float v;
    int cv;
    block_max_count(arr, sm, n, below, tid, v, cv);
    if (cv == 0) break;  // (not reached: the columns' mass reaches thr)
    const unsigned long long mv =
        (unsigned long long)__float2ull_rn(exp2_scaled(v, scale, M) * kFix);
    const double need = thr - double(before);  // > 0
    if (double(before) + double(mv) * double(cv) >= thr || mv == 0ull) {
      // kept: the first k columns of the run, k = ceil(need / mv) (at least 1)
      long long k = mv == 0ull ? cv : (long long)ceil(need / double(mv));
      k = k < 1 ? 1 : (k > cv ? cv : k);
      // the k-th smallest column among the run (ranks by counting)
      for (int i = tid; i < n; i += kNT) {
        const Cand e = arr[i];
        if (e.v != v) continue;
        int rank = 0;
        for (int j = 0; j < n; ++j) rank += (arr[j].v == v && arr[j].c < e.c);
        if (rank == k - 1) sm.cross = e.c;  // exactly one thread
      }
      __syncthreads();
      tau = v;
      tau_col = sm.cross;
      __syncthreads();
      return;
    }
    before += mv * (unsigned long long)cv;
    below = v;
  }
}

// The kept set of a nucleus row from one pass over its logits, when the cut
// lies among the columns within kCandDelta log2 units of the row maximum M
// (a column there weighs at least 2^-kCandDelta of the maximum's mass): those
// columns are gathered in shared memory, their masses (40-bit fixed point)
// binned by delta at 1/32 log2 unit, and the bucket where the running mass,
// largest logits first, reaches top_p of the row's total (from the partials)
// is walked by value. Every column above zc is a candidate, so the walk over
// the candidates in rank order is the walk over the whole row down to zc, and
// a cut reached among them is the row's cut. Candidates that overflow the
// buffer at the first bar are gathered again at a lower one (below). Returns
// false -- and the caller runs the histogram levels over the whole row -- when
// the candidates still overflow the buffer, their mass stays below the cut, or
// the crossing bucket holds more than kCross of them. On true, sm.cacc holds
// the kept masses per chunk.
// Every thread calls and gets the same result.
__device__ bool candidate_cut(const Partial* part, NucSmem& sm, const char* row, int dt, int V,
                              int nvec, int vec, int nch, float M, float scale, float top_p,
                              float& tau, int& tau_col) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // the row's total 2^(z * scale - M), compensated, from the partials
  F2 T = {0.f, 0.f};
  for (int c = tid; c < nch; c += kNT) {
    const Partial q = part[c];
    if (q.m > -INFINITY) T = f2_add(T, F2{__fmul_rn(q.s, ex2_approx(q.m - M)), 0.f});
  }
  T = block_sum_f2(T, sm, lane, warp);
  const double Td = double(T.hi) + double(T.lo);
  if (!(Td > 0.0) || !isfinite(Td)) return false;
  const double thr = double(top_p) * Td * double(kFix);
  // Candidates: z > zc, zc = (M - bar) / scale. The first pass uses the bar
  // kCandDelta; when its candidates overflow the buffer, a second pass takes
  // the largest lower whole bar whose candidates, estimated from the ones the
  // buffer holds, fit (a row whose cut lies below that bar is still settled;
  // the others take the histogram levels).
  float bar = kCandDelta;
  bool over = false;
  for (int attempt = 0; attempt < 2; ++attempt) {
    const float zc = __fdiv_rn(__fsub_rn(M, bar), scale);  // candidates: z > zc
    if (tid == 0) {
      sm.n_gc = 0;
      sm.cross = -1;
    }
    if (tid < kNW) sm.wn[tid] = 0;
    if (tid < kUnitBins) sm.ucnt[tid] = 0.f;
    for (int c = tid; c < nch; c += kNT) sm.cacc[c] = 0ull;
    for (int i = tid; i < kCandBuckets; i += kNT) sm.mass[i] = 0ull;
    __syncthreads();
    // ------------------------------------ one pass over the row: the candidates
    // A vector holding a logit above zc has its candidates appended at once by
    // its lane (the row is not read again: the rows in flight across the GPU
    // exceed L2), each warp to its own region of the buffer (kRegion entries;
    // the columns are spread over the warps, so a region overflows only when
    // the whole buffer nearly would).
    Cand* region = sm.gz + warp * kRegion;
    auto take = [&](float z, int x) {
      const int i = atomicAdd(&sm.wn[warp], 1);
      if (i < kRegion) region[i] = Cand{z, x};
    };
    scan_row<kNT, 8>(reinterpret_cast<const uint4*>(row), nvec, dt, zc, tid,
                     [&](int v, const uint4& w) { vector_candidates(w, dt, v, zc, take); });
    for (int x = nvec * vec + tid; x < V; x += kNT) {  // the ragged tail
      const float z = load_dt(row, dt, x);
      if (z > zc) take(z, x);
    }
    __syncthreads();
    over = false;
#pragma unroll
    for (int x = 0; x < kNW; ++x) over |= sm.wn[x] > kRegion;
    if (!over || attempt == 1) break;
    // The buffer holds the first candidates of each warp's columns, a sample of
    // all of them whose spread in delta (per whole log2 unit) estimates theirs:
    // the largest whole bar below this one whose estimated candidates fit with
    // room to spare in every warp's region.
    for (int x = 0; x < kNW; ++x) {
      const int held = min(sm.wn[x], kRegion);
      const float weight = float(sm.wn[x]) / float(max(held, 1));  // candidates per held one
      for (int i = tid; i < held; i += kNT) {
        const float dd = __fsub_rn(M, __fmul_rn(sm.gz[x * kRegion + i].v, scale));
        atomicAdd(&sm.ucnt[min(kUnitBins - 1, max(0, int(dd)))], weight);
      }
    }
    __syncthreads();
    float nb = 0.f, below = 0.f;
    for (int d = 0; d < int(bar); ++d) {
      below += sm.ucnt[d];
      if (below > float(kRetryCands)) break;
      nb = float(d + 1);
    }
    __syncthreads();  // every thread has read the counts before they are cleared
    if (!(nb >= kMinBar && nb < bar)) break;
    bar = nb;
  }
  if (over) return false;
  int ng = 0;
#pragma unroll
  for (int x = 0; x < kNW; ++x) ng += sm.wn[x];
  // every gathered candidate, region by region
  auto for_cands = [&](auto&& fn) {
    for (int x = 0; x < kNW; ++x) {
      const int n = sm.wn[x];
      for (int i = tid; i < n; i += kNT) fn(sm.gz[x * kRegion + i]);
    }
  };

  // ------------------------ candidate masses binned by delta (1/32 log2 unit)
  auto fixm = [&](float z) {
    return (unsigned long long)__float2ull_rn(exp2_scaled(z, scale, M) * kFix);
  };
  auto bucket = [&](float z) {  // non-increasing in z
    const float f = __fsub_rn(M, __fmul_rn(z, scale)) * kBucketsPerUnit;
    return f > 0.f ? min(kCandBuckets - 1, int(f)) : 0;
  };
  for_cands([&](const Cand& e) { atomicAdd(&sm.mass[bucket(e.v)], fixm(e.v)); });
  __syncthreads();
  // the first bucket whose inclusive running mass reaches thr (thread t owns a
  // contiguous run of buckets)
  constexpr int kPer = (kCandBuckets + kNT - 1) / kNT;
  const int b0 = tid * kPer, b1 = min(kCandBuckets, b0 + kPer);
  unsigned long long loc = 0ull;
  for (int i = b0; i < b1; ++i) loc += sm.mass[i];
  unsigned long long incl = loc;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) sm.wsum[warp] = incl;
  __syncthreads();
  unsigned long long wbase = 0ull;
#pragma unroll
  for (int x = 0; x < kNW; ++x)
    if (x < warp) wbase += sm.wsum[x];
  unsigned long long run = wbase + incl - loc;
  for (int i = b0; i < b1; ++i) {
    const unsigned long long nx = run + sm.mass[i];
    if (double(nx) >= thr && double(run) < thr) sm.cross = i;  // one bucket at most
    run = nx;
  }
  __syncthreads();
  const int cb = sm.cross;
  if (cb < 0) return false;  // the candidates' mass stays below the cut
  unsigned long long pre = 0ull;
  for (int i = tid; i < cb; i += kNT) pre += sm.mass[i];
  const unsigned long long before = block_sum_u64(pre, sm, lane, warp);
  // the crossing bucket's candidates, apart
  for_cands([&](const Cand& e) {
    if (bucket(e.v) == cb) {
      const int j = atomicAdd(&sm.n_gc, 1);
      if (j < kCross) sm.gc[j] = e;
    }
  });
  __syncthreads();
  const int nc = sm.n_gc;
  if (nc > kCross) return false;
  if (nc <= 32) {
    // one lane per candidate: a candidate is kept when the mass ranked before
    // it (larger logit, then smaller column) is below thr; the last kept one
    // has the most mass before it (every candidate's mass is positive)
    if (warp == 0) {
      const bool has = lane < nc;
      const Cand e = has ? sm.gc[lane] : Cand{-INFINITY, 0x7fffffff};
      const unsigned long long me = has ? fixm(e.v) : 0ull;
      unsigned long long pm = 0ull;
      for (int j = 0; j < nc; ++j) {
        const float vj = __shfl_sync(0xffffffffu, e.v, j);
        const int cj = __shfl_sync(0xffffffffu, e.c, j);
        const unsigned long long mj = __shfl_sync(0xffffffffu, me, j);
        if (vj > e.v || (vj == e.v && cj < e.c)) pm += mj;
      }
      const bool kept = has && double(before + pm) < thr;
      unsigned long long key = kept ? pm + 1ull : 0ull;
      int src = lane;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long ok = __shfl_xor_sync(0xffffffffu, key, o);
        const int os = __shfl_xor_sync(0xffffffffu, src, o);
        if (ok > key || (ok == key && os < src)) {
          key = ok;
          src = os;
        }
      }
      if (lane == src) {
        sm.tau_v = e.v;
        sm.tau_c = e.c;
      }
    }
    __syncthreads();
    tau = sm.tau_v;
    tau_col = sm.tau_c;
  } else {
    walk_runs(sm.gc, nc, before, thr, sm, M, scale, tau, tau_col);
  }
  // the kept candidates join their chunks
  for_cands([&](const Cand& e) {
    if (e.v > tau || (e.v == tau && e.c <= tau_col)) atomicAdd(&sm.cacc[e.c / kChunk], fixm(e.v));
  });
  return ng > 0;
}

// Shared memory of one warp of nucleus_warp_kernel (about 7.7 KB).
struct NucWarpSmem {
  Cand cand[kWCap];
  unsigned long long mass[kWBuckets];
  Cand gc[32];
  unsigned long long cacc[kWChunks];
  int n, ngc;
};

// The kept set of a narrow nucleus row (at most kWarpRowMax columns), one warp
// per row: the candidate way of candidate_cut at warp scale -- the columns
// within kWCandDelta log2 units of the row maximum gathered, their fixed-point
// masses binned by delta at 1/32 log2 unit, the crossing bucket ranked one
// candidate per lane. A row whose candidates overflow kWCap, do not reach the
// cut or put more than 32 in the crossing bucket gets head n = -1 and is left
// to nucleus_kernel.
__global__ void __launch_bounds__(kWWarps * 32, 3) nucleus_warp_kernel(KeptArgs a) {
  extern __shared__ __align__(16) char wsm_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  NucWarpSmem& sm = reinterpret_cast<NucWarpSmem*>(wsm_raw)[warp];
  const int64_t rows_d = (a.d.nucleus && a.d.V <= kWarpRowMax) ? a.rows_d : 0;
  const int64_t rows_t = (a.t.nucleus && a.t.V <= kWarpRowMax) ? a.rows_t : 0;
  grid_dependency_wait();  // the partials (and the need flags) come from earlier kernels
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int64_t w = int64_t(blockIdx.x) * kWWarps + warp; w < rows_d + rows_t;
       w += int64_t(gridDim.x) * kWWarps) {
    const bool tgt = w >= rows_d;
    const int64_t r = tgt ? w - rows_d : w;
    const RowSet& S = tgt ? a.t : a.d;
    if (!tgt && S.need && S.need[r] == 0) continue;
    const int dt = tgt ? a.dt_t : a.dt_d;
    const float top_p = tgt ? a.top_p_t : a.top_p_d;
    KeptHead* head = (tgt ? a.head_t : a.head_d) + r;
    float* um = (tgt ? a.um_t : a.um_d) + r * S.nch;
    const int V = S.V, nch = S.nch;
    const float scale = S.scale;
    const char* row = S.data + r * S.stride_bytes;
    const int vec = dt == TT_F32 ? 4 : 8;
    const int nvec = V / vec;
    const Partial* part = S.part + r * nch;
    // the row maximum and total from the partials (compensated)
    float M = -INFINITY;
    for (int c = lane; c < nch; c += 32) M = fmaxf(M, part[c].m);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if (!isfinite(M)) {
      if (lane == 0) *head = KeptHead{NAN, 0, NAN, -1, M, 0.f};
      continue;
    }
    F2 T = {0.f, 0.f};
    for (int c = lane; c < nch; c += 32) {
      const Partial q = part[c];
      if (q.m > -INFINITY) T = f2_add(T, F2{__fmul_rn(q.s, ex2_approx(q.m - M)), 0.f});
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
      T = f2_add(T, F2{__shfl_xor_sync(0xffffffffu, T.hi, o), __shfl_xor_sync(0xffffffffu, T.lo, o)});
    const double Td = double(T.hi) + double(T.lo);
    if (!(Td > 0.0) || !isfinite(Td)) {
      if (lane == 0) head->n = -1;
      continue;
    }
    const double thr = double(top_p) * Td * double(kFix);
    const float zc = __fdiv_rn(__fsub_rn(M, kWCandDelta), scale);  // candidates: z > zc
    auto fixm = [&](float z) {
      return (unsigned long long)__float2ull_rn(exp2_scaled(z, scale, M) * kFix);
    };
    auto bucket = [&](float z) {  // non-increasing in z
      const float f = __fsub_rn(M, __fmul_rn(z, scale)) * kBucketsPerUnit;
      return f > 0.f ? min(kWBuckets - 1, int(f)) : 0;
    };
    if (lane == 0) {
      sm.n = 0;
      sm.ngc = 0;
    }
    for (int i = lane; i < kWBuckets; i += 32) sm.mass[i] = 0ull;
    if (lane < kWChunks) sm.cacc[lane] = 0ull;
    __syncwarp();
    // one pass over the row; a vector holding candidates has them appended at
    // once by its lane
    auto take = [&](float z, int x) {
      const int i = atomicAdd(&sm.n, 1);
      if (i < kWCap) sm.cand[i] = Cand{z, x};
    };
    scan_row<32, 8>(reinterpret_cast<const uint4*>(row), nvec, dt, zc, lane,
                    [&](int v, const uint4& w) { vector_candidates(w, dt, v, zc, take); });
    for (int x = nvec * vec + lane; x < V; x += 32) {  // the ragged tail
      const float z = load_dt(row, dt, x);
      if (z > zc) take(z, x);
    }
    __syncwarp();
    const int n = sm.n;
    if (n > kWCap || n == 0) {
      if (lane == 0) head->n = -1;
      __syncwarp();
      continue;
    }
    for (int i = lane; i < n; i += 32) {
      const Cand e = sm.cand[i];
      atomicAdd(&sm.mass[bucket(e.v)], fixm(e.v));
    }
    __syncwarp();
    // the first bucket whose inclusive running mass reaches thr (lane l owns a
    // contiguous run of buckets)
    constexpr int kPer = (kWBuckets + 31) / 32;
    const int b0 = lane * kPer, b1 = min(kWBuckets, b0 + kPer);
    unsigned long long loc = 0ull;
    for (int i = b0; i < b1; ++i) loc += sm.mass[i];
    unsigned long long incl = loc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    unsigned long long run = incl - loc, before = 0ull;
    int cb = kWBuckets;
    for (int i = b0; i < b1; ++i) {
      const unsigned long long nx = run + sm.mass[i];
      if (double(nx) >= thr && double(run) < thr) {
        cb = i;
        before = run;
      }
      run = nx;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int ocb = __shfl_xor_sync(0xffffffffu, cb, o);
      const unsigned long long ob = __shfl_xor_sync(0xffffffffu, before, o);
      if (ocb < cb) {
        cb = ocb;
        before = ob;
      }
    }
    if (cb >= kWBuckets) {  // the candidates' mass stays below the cut
      if (lane == 0) head->n = -1;
      __syncwarp();
      continue;
    }
    for (int i = lane; i < n; i += 32) {
      const Cand e = sm.cand[i];
      if (bucket(e.v) == cb) {
        const int j = atomicAdd(&sm.ngc, 1);
        if (j < 32) sm.gc[j] = e;
      }
    }
    __syncwarp();
    const int nc = sm.ngc;
    if (nc > 32) {
      if (lane == 0) head->n = -1;
      __syncwarp();
      continue;
    }
    // one lane per candidate of the crossing bucket (see candidate_cut)
    const bool has = lane < nc;
    const Cand e = has ? sm.gc[lane] : Cand{-INFINITY, 0x7fffffff};
    const unsigned long long me = has ? fixm(e.v) : 0ull;
    unsigned long long pm = 0ull;
    for (int j = 0; j < nc; ++j) {
      const float vj = __shfl_sync(0xffffffffu, e.v, j);
      const int cj = __shfl_sync(0xffffffffu, e.c, j);
      const unsigned long long mj = __shfl_sync(0xffffffffu, me, j);
      if (vj > e.v || (vj == e.v && cj < e.c)) pm += mj;
    }
    const bool kept = has && double(before + pm) < thr;
    unsigned long long key = kept ? pm + 1ull : 0ull;
    int src = lane;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long ok = __shfl_xor_sync(0xffffffffu, key, o);
      const int os = __shfl_xor_sync(0xffffffffu, src, o);
      if (ok > key || (ok == key && os < src)) {
        key = ok;
        src = os;
      }
    }
    const float tau = __shfl_sync(0xffffffffu, e.v, src);
    const int tau_col = __shfl_sync(0xffffffffu, e.c, src);
    // the kept candidates join their chunks; the header
    for (int i = lane; i < n; i += 32) {
      const Cand c = sm.cand[i];
      if (c.v > tau || (c.v == tau && c.c <= tau_col))
        atomicAdd(&sm.cacc[c.c / kChunk], fixm(c.v));
    }
    __syncwarp();
    unsigned long long tot = lane < nch ? sm.cacc[lane] : 0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    const double Sd = double(tot) / double(kFix);  // kept normaliser relative to 2^M
    if (lane < nch) um[lane] = float(double(sm.cacc[lane]) / double(kFix) / Sd);
    if (lane == 0) {
      const float lse = float((double(M) + log2(Sd)) * 0.6931471805599453);
      *head = KeptHead{lse, 1, tau, tau_col, M, float(1.0 / Sd)};
    }
    __syncwarp();  // shared memory is reused by the warp's next row
  }
}

// One CTA per nucleus row: every row of a family wider than kWarpRowMax, and
// the rows of a narrower family that nucleus_warp_kernel left (head n = -1),
// found 256 rows at a time. Tiles of draft rows, then of target rows,
// grid-stride.
__global__ void __launch_bounds__(kNT, 3) nucleus_kernel(KeptArgs a) {
  extern __shared__ __align__(16) char nsm_raw[];
  NucSmem& sm = *reinterpret_cast<NucSmem*>(nsm_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t rows_d = a.d.nucleus ? a.rows_d : 0, rows_t = a.t.nucleus ? a.rows_t : 0;
  const int tsz_d = a.d.V <= kWarpRowMax ? kNT : 1, tsz_t = a.t.V <= kWarpRowMax ? kNT : 1;
  const int64_t nt_d = (rows_d + tsz_d - 1) / tsz_d, nt_t = (rows_t + tsz_t - 1) / tsz_t;
  grid_dependency_wait();  // the partials (and the need flags) come from earlier kernels
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  for (int64_t tile = blockIdx.x; tile < nt_d + nt_t; tile += gridDim.x) {
  const bool tgt = tile >= nt_d;
  const int tsz = tgt ? tsz_t : tsz_d;
  const int64_t r0 = (tgt ? tile - nt_d : tile) * tsz;
  int n_todo = 1;
  if (tsz > 1) {  // the narrow rows the warp kernel could not settle
    __syncthreads();
    if (tid == 0) sm.n_todo = 0;
    __syncthreads();
    const int64_t rr = r0 + tid;
    const RowSet& SF = tgt ? a.t : a.d;
    const KeptHead* hf = tgt ? a.head_t : a.head_d;
    if (rr < (tgt ? rows_t : rows_d) && (tgt || !SF.need || SF.need[rr] != 0) && hf[rr].n == -1)
      sm.todo[atomicAdd(&sm.n_todo, 1)] = tid;
    __syncthreads();
    n_todo = sm.n_todo;
  }
  for (int k = 0; k < n_todo; ++k) {
    const int64_t r = tsz > 1 ? r0 + sm.todo[k] : r0;
    const RowSet& S = tgt ? a.t : a.d;
    if (!tgt && S.need && S.need[r] == 0) continue;
    const int dt = tgt ? a.dt_t : a.dt_d;
    const float top_p = tgt ? a.top_p_t : a.top_p_d;
    KeptHead* head = (tgt ? a.head_t : a.head_d) + r;
    float* um = (tgt ? a.um_t : a.um_d) + r * S.nch;
    const int V = S.V, nch = S.nch;
    const float scale = S.scale;
    const char* row = S.data + r * S.stride_bytes;
    const int vec = dt == TT_F32 ? 4 : 8;  // logits per 16-byte vector
    const int nvec = V / vec;              // whole vectors (rows start on 16 bytes)

    // the row maximum from the partials (nucleus rows' partials hold every column)
    float M = -INFINITY;
    for (int c = tid; c < nch; c += kNT) M = fmaxf(M, S.part[r * nch + c].m);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    __syncthreads();
    if (lane == 0) sm.wmax[warp] = __float_as_uint(M) ^ (M < 0.f ? 0xffffffffu : 0x80000000u);
    __syncthreads();
    {
      unsigned long long best = 0;
#pragma unroll
      for (int x = 0; x < kNW; ++x) best = max(best, sm.wmax[x]);
      const uint32_t key = uint32_t(best);
      M = __uint_as_float(key & 0x80000000u ? key ^ 0x80000000u : ~key);
    }
    if (!isfinite(M)) {
      if (tid == 0) *head = KeptHead{NAN, 0, NAN, -1, M, 0.f};
      continue;
    }

    // every column once per pass, 16-byte vectors and the ragged tail
    auto for_each = [&](auto&& fn) {
      for (int v = tid; v < nvec; v += kNT) {
        const uint4 w4 = __ldg(reinterpret_cast<const uint4*>(row) + v);
        const uint32_t ww[4] = {w4.x, w4.y, w4.z, w4.w};
        if (dt == TT_F32) {
#pragma unroll
          for (int q = 0; q < 4; ++q) fn(v * 4 + q, __uint_as_float(ww[q]));
        } else {
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            fn(v * 8 + 2 * q, __uint_as_float(ww[q] << 16));
            fn(v * 8 + 2 * q + 1, __uint_as_float(ww[q] & 0xffff0000u));
          }
        }
      }
      for (int x = nvec * vec + tid; x < V; x += kNT) fn(x, load_dt(row, dt, x));
    };
    auto delta_of = [&](float z) { return __fsub_rn(M, __fmul_rn(z, scale)); };
    // mass 2^(z * scale - M) in 40-bit fixed point (the exponent split exactly)
    auto fixm = [&](float z) {
      return (unsigned long long)__float2ull_rn(exp2_scaled(z, scale, M) * kFix);
    };

    float tau = -INFINITY;
    int tau_col = 0x7fffffff;  // all kept: every column ranks before (tau, tau_col)
    const bool settled = candidate_cut(S.part + r * nch, sm, row, dt, V, nvec, vec, nch, M,
                                       scale, top_p, tau, tau_col);
    if (!settled) {
    // ------------------------------------- the crossing bucket, level by level
    Path cross;
    int level = 0;
    unsigned long long total = 0ull;
    double thr = 0.0;
    bool all_kept = false;
    for (int c = tid; c < nch; c += kNT) sm.cacc[c] = 0ull;
    if (tid == 0) {
      sm.before = 0ull;
      sm.n_gz = 0;
    }
    __syncthreads();
    cross.b[0] = cross.b[1] = cross.b[2] = 0;
    for (; level < kLevels; ++level) {
      for (int i = tid; i < kBuckets; i += kNT) {
        sm.cnt[i] = 0u;
        sm.mass[i] = 0ull;
      }
      __syncthreads();
      for_each([&](int x, float z) {
        const float d = delta_of(z);
        const Path p = bucket_path(d);
        if (p.b[0] < 0) return;
        if (level > 0 && path_cmp(p, cross, level - 1) != 0) return;
        atomicAdd(&sm.cnt[p.b[level]], 1u);
        atomicAdd(&sm.mass[p.b[level]], fixm(z));
      });
      __syncthreads();
      // running mass over the buckets (thread t owns a contiguous run of them)
      constexpr int kPer = (kBuckets + kNT - 1) / kNT;
      const int b0 = tid * kPer, b1 = min(kBuckets, b0 + kPer);
      unsigned long long loc = 0ull;
      for (int i = b0; i < b1; ++i) loc += sm.mass[i];
      unsigned long long incl = loc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long n = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += n;
      }
      __syncthreads();
      if (lane == 31) sm.wsum[warp] = incl;
      __syncthreads();
      unsigned long long wbase = 0ull, all = 0ull;
#pragma unroll
      for (int x = 0; x < kNW; ++x) {
        if (x < warp) wbase += sm.wsum[x];
        all += sm.wsum[x];
      }
      const unsigned long long before0 = sm.before;
      if (level == 0) {
        total = all;
        thr = double(top_p) * double(total);
        if (tid == 0) sm.cross = -1;
      } else if (tid == 0) {
        sm.cross = -1;
      }
      __syncthreads();
      // the first bucket whose inclusive running mass reaches thr
      unsigned long long run = before0 + wbase + incl - loc;
      for (int i = b0; i < b1; ++i) {
        const unsigned long long nx = run + sm.mass[i];
        if (double(nx) >= thr && double(run) < thr) atomicMax(&sm.cross, i);
        run = nx;
      }
      __syncthreads();
      const int cb = sm.cross;
      if (cb < 0) {  // the counted columns never reach the cut: all are kept
        all_kept = true;
        break;
      }
      cross.b[level] = cb;
      // mass before the crossing bucket
      unsigned long long pre = 0ull;
      for (int i = tid; i < cb; i += kNT) pre += sm.mass[i];
      pre = block_sum_u64(pre, sm, lane, warp);
      if (tid == 0) sm.before = before0 + pre;
      const unsigned int ccount = sm.cnt[cb];
      __syncthreads();
      if (ccount <= unsigned(kRefine) || level == kLevels - 1) break;
    }
    if (level == kLevels) level = kLevels - 1;

    // --------------------- gather the crossing bucket; chunk masses before it
    for_each([&](int x, float z) {
      const float d = delta_of(z);
      const Path p = bucket_path(d);
      if (p.b[0] < 0) return;
      const int c = all_kept ? -1 : path_cmp(p, cross, level);
      if (c < 0) {
        atomicAdd(&sm.cacc[x / kChunk], fixm(z));
      } else if (c == 0) {
        const int i = atomicAdd(&sm.n_gz, 1);
        if (i < kGather) sm.gz[i] = Cand{z, x};
      }
    });
    __syncthreads();
    const int ng = sm.n_gz;
    if (!all_kept) {
      if (ng <= kGather) {
        walk_runs(sm.gz, ng, sm.before, thr, sm, M, scale, tau, tau_col);
        // the kept columns of the crossing bucket join their chunks
        for (int i = tid; i < ng; i += kNT) {
          const Cand e = sm.gz[i];
          if (e.v > tau || (e.v == tau && e.c <= tau_col))
            atomicAdd(&sm.cacc[e.c / kChunk], fixm(e.v));
        }
      } else {
        // a crossing run of more than kGather tied columns (the last level holds
        // one delta per bucket): the same walk with passes over the row
        unsigned long long before = sm.before;
        float below = INFINITY;
        for (;;) {
          float v = -INFINITY;
          for_each([&](int x, float z) {
            const Path p = bucket_path(delta_of(z));
            if (p.b[0] >= 0 && path_cmp(p, cross, level) == 0 && z < below) v = fmaxf(v, z);
          });
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
          __syncthreads();
          if (lane == 0) sm.wmax[warp] = __float_as_uint(v) ^ (v < 0.f ? 0xffffffffu : 0x80000000u);
          __syncthreads();
          unsigned long long best = 0;
#pragma unroll
          for (int x = 0; x < kNW; ++x) best = max(best, sm.wmax[x]);
          const uint32_t key = uint32_t(best);
          v = __uint_as_float(key & 0x80000000u ? key ^ 0x80000000u : ~key);
          if (!(v > -INFINITY)) break;
          int cv = 0;
          for_each([&](int x, float z) { cv += z == v; });
          cv = int(block_sum_u64((unsigned long long)cv, sm, lane, warp));
          const unsigned long long mv = fixm(v);
          if (double(before) + double(mv) * double(cv) >= thr || mv == 0ull) {
            long long k = mv == 0ull ? cv : (long long)ceil((thr - double(before)) / double(mv));
            k = k < 1 ? 1 : (k > cv ? cv : k);
            // the k-th column holding v, in column order: thread t scans columns
            // t * seg .. (t + 1) * seg
            const int seg = (V + kNT - 1) / kNT;
            const int x0 = tid * seg, x1 = min(V, x0 + seg);
            int mine = 0;
            for (int x = x0; x < x1; ++x) mine += load_dt(row, dt, x) == v;
            int incl = mine;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
              const int n = __shfl_up_sync(0xffffffffu, incl, o);
              if (lane >= o) incl += n;
            }
            __syncthreads();
            if (lane == 31) sm.wcnt[warp] = incl;
            __syncthreads();
            int base = 0;
            for (int x = 0; x < warp; ++x) base += sm.wcnt[x];
            const long long first = base + incl - mine;  // runs before this thread's
            if (k > first && k <= first + mine) {
              long long seen = first;
              for (int x = x0; x < x1; ++x)
                if (load_dt(row, dt, x) == v && ++seen == k) {
                  sm.cross = x;
                  break;
                }
            }
            __syncthreads();
            tau = v;
            tau_col = sm.cross;
            break;
          }
          before += mv * (unsigned long long)cv;
          below = v;
        }
        // the kept columns of the crossing bucket join their chunks
        for_each([&](int x, float z) {
          const float d = delta_of(z);
          const Path p = bucket_path(d);
          if (p.b[0] >= 0 && path_cmp(p, cross, level) == 0 &&
              (z > tau || (z == tau && x <= tau_col)))
            atomicAdd(&sm.cacc[x / kChunk], fixm(z));
        });
      }
    }
    }  // !settled
    __syncthreads();
    // ---------------------------------------------- header and chunk masses
    unsigned long long tot = 0ull;
    for (int c = tid; c < nch; c += kNT) tot += sm.cacc[c];
    tot = block_sum_u64(tot, sm, lane, warp);
    const double Sd = double(tot) / double(kFix);  // kept normaliser relative to 2^M
    const float inv_s = float(1.0 / Sd);
    for (int c = tid; c < nch; c += kNT) um[c] = float(double(sm.cacc[c]) / double(kFix) / Sd);
    if (tid == 0) {
      const float lse = float((double(M) + log2(Sd)) * 0.6931471805599453);
      *head = KeptHead{lse, tot > 0ull ? 1 : 0, tau, tau_col, M, inv_s};
    }
    __syncthreads();  // shared memory is reused by the next row
  }
  }
}

// The decision over nucleus target rows (one CTA per request): p(t_j) from
// each row's kept set, the accept test (Alg. 2 / Alg. 4), and the residual of
// row a (one-hot q: the kept set with t_a's probability lowered by q_hat) or
// the bonus row, drawn by inverse CDF in column order at two levels: the chunk
// from the kept chunk masses, the column from that chunk's logits re-read.
__global__ void __launch_bounds__(kNT) decide_nucleus_kernel(DecideArgs a) {
  __shared__ float s_p[TT_MAX_M];
  __shared__ int s_a, s_nf, s_pick, s_last, s_chunk;
  __shared__ F2 s_rel;
  __shared__ F2 wtot[kNW], wpre[kNW + 1];
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
  if (tid == 0) {
    s_a = m;
    s_nf = 0;
    s_pick = -1;
    s_last = -1;
    s_chunk = -1;
  }
  int bad = 0;
  if (st == 0)
    for (int j = tid; j < m; j += kNT) {
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
  if (a.err && a.err[0] == a.epoch) st = a.err[1];  // the row pass failed
  if (st != 0) {
    if (tid == 0) {
      a.accepted[b] = 0;
      a.next_token[b] = -1;
      a.status[b] = st;
    }
    return;
  }
  const RowSet& T = a.t;
  const int V = T.V, nch = T.nch;
  const float scale = T.scale;
  // target rows 0..m: p(t_j) = 2^(z * scale - M) / S when t_j is kept, lse
  for (int j = tid; j <= m; j += kNT) {
    const int64_t row = int64_t(t0) + b + j;
    const KeptHead h = a.head_t[row];
    if (h.n == 0) s_nf = 1;
    if (j < m) {
      const int c = a.target_cols[t0 + j];
      const float z = load_dt(T.data + row * T.stride_bytes, a.dt_t, c);
      const bool kept = z > h.tau || (z == h.tau && c <= h.tau_col);
      const float p = kept ? exp2_scaled(z, scale, h.M) * h.inv_s : 0.f;
      s_p[j] = p;
      if (a.p_hat) a.p_hat[t0 + j] = p;
    }
    if (a.lse) a.lse[row] = h.lse;
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
  for (int j = tid; j < m; j += kNT) {
    const float u = float(philox_uniform(a.seed, uint64_t(j), 0, req));
    if (!(u * a.q_hat_in[t0 + j] < s_p[j])) atomicMin(&s_a, j);
  }
  __syncthreads();
  const int acc = s_a;
  const int64_t row = int64_t(t0) + b + acc;
  const KeptHead h = a.head_t[row];
  const char* trow = T.data + row * T.stride_bytes;
  const float* um = a.um_t + row * nch;
  const int t = acc < m ? a.target_cols[t0 + acc] : -1;
  const float pt = acc < m ? s_p[acc] : 0.f;
  float rt = acc < m ? fmaxf(0.f, pt - a.q_hat_in[t0 + acc]) : 0.f;
  const int ct = t >= 0 ? t / kChunk : -1;
  // coarse level: chunk masses (thread tid owns chunks tid * per ..)
  const int per = (nch + kNT - 1) / kNT;
  const int c0 = min(nch, tid * per), c1 = min(nch, c0 + per);
  auto block_prefix = [&](F2 v, F2& excl, F2& total) {
    F2 incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const F2 n = shfl_up_f2(incl, o, 32);
      if (lane >= o) incl = f2_add(n, incl);
    }
    const F2 prev = shfl_up_f2(incl, 1, 32);
    excl = lane == 0 ? F2{0.f, 0.f} : prev;
    __syncthreads();
    if (lane == 31) wtot[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      F2 wi = lane < kNW ? wtot[lane] : F2{0.f, 0.f};
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const F2 n = shfl_up_f2(wi, o, 32);
        if (lane >= o) wi = f2_add(n, wi);
      }
      const F2 wp = shfl_up_f2(wi, 1, 32);
      if (lane <= kNW) wpre[lane] = lane == 0 ? F2{0.f, 0.f} : wp;
    }
    __syncthreads();
    excl = f2_add(wpre[warp], excl);
    total = wpre[kNW];
  };
  // the residual's chunk masses: t's chunk loses p_t and gains r_t; with no
  // mass left, the row itself
  auto chunk_mass = [&](int c, bool resid) -> float {
    float x = um[c];
    if (resid && c == ct) x = fmaxf(0.f, x - pt + rt);
    return x;
  };
  F2 loc = {0.f, 0.f};
  for (int c = c0; c < c1; ++c) loc = f2_add(loc, F2{chunk_mass(c, true), 0.f});
  F2 excl, Z;
  block_prefix(loc, excl, Z);
  bool resid = true;
  if (!(Z.hi > 0.f)) {  // degenerate residual: the row itself
    resid = false;
    rt = pt;
    loc = {0.f, 0.f};
    for (int c = c0; c < c1; ++c) loc = f2_add(loc, F2{chunk_mass(c, false), 0.f});
    block_prefix(loc, excl, Z);
  }
  const float u2 = float(philox_uniform(a.seed, uint64_t(acc), 1, req));
  const F2 th = f2_mul_f(Z, u2);
  {
    F2 cum = excl;
    int last = -1;
    for (int c = c0; c < c1; ++c) {
      const float x = chunk_mass(c, resid);
      const F2 nx = f2_add(cum, F2{x, 0.f});
      if (x > 0.f) {
        last = c;
        if (!f2_lt(th, cum) && f2_lt(th, nx)) {
          s_chunk = c;
          s_rel = f2_add(th, F2{-cum.hi, -cum.lo});
        }
      }
      cum = nx;
    }
    if (last >= 0) atomicMax(&s_last, last);
  }
  __syncthreads();
  F2 rel;
  int chunk = s_chunk;
  if (chunk >= 0) {
    rel = s_rel;
  } else {  // theta at the very top by rounding: the last chunk with mass
    chunk = max(0, s_last);
    rel = {INFINITY, 0.f};
  }
  __syncthreads();
  if (tid == 0) s_last = -1;
  // fine level: the chunk's kept columns in column order, 8 per thread
  const int x0 = chunk * kChunk + tid * 8;
  float r[8];
  F2 run = {0.f, 0.f};
  int last_pos = -1;
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const int x = x0 + q;
    float v = 0.f;
    if (x < V) {
      const float z = load_dt(trow, a.dt_t, x);
      const bool kept = z > h.tau || (z == h.tau && x <= h.tau_col);
      if (kept) v = x == t ? rt : exp2_scaled(z, scale, h.M) * h.inv_s;
    }
    if (v > 0.f) last_pos = x;
    r[q] = v;
    run = f2_add(run, F2{v, 0.f});
  }
  F2 ex2, tot2;
  block_prefix(run, ex2, tot2);
  const F2 in2 = f2_add(ex2, run);
  if (!f2_lt(rel, ex2) && f2_lt(rel, in2)) {
    F2 c = ex2;
    int pick = last_pos;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
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
    const int pick = s_pick >= 0 ? s_pick : s_last;
    a.accepted[b] = acc;
    a.next_token[b] = pick;
    a.status[b] = pick >= 0 ? 0 : TT_REQ_NOT_FINITE;
  }
}

static_assert(3 * (sizeof(NucSmem) + 1024) <= 227 * 1024, "three nucleus CTAs fit on an SM");
static_assert(3 * (kWWarps * sizeof(NucWarpSmem) + 1024) <= 227 * 1024,
              "three warp-kernel CTAs fit on an SM");

}  // namespace

cudaError_t preload_nucleus() {
  cudaError_t e = cudaFuncSetAttribute(nucleus_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(sizeof(NucSmem)));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(nucleus_warp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           int(kWWarps * sizeof(NucWarpSmem)));
  if (e != cudaSuccess) return e;
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, decide_nucleus_kernel);
}

cudaError_t launch_decide_nucleus(const DecideArgs& args, cudaStream_t stream, bool pdl) {
  if (args.B == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(args.B));
  cfg.blockDim = dim3(kNT);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decide_nucleus_kernel, args);
}

cudaError_t launch_nucleus(const KeptArgs& args, cudaStream_t stream, int sm_count, bool pdl) {
  const int64_t rows = (args.d.nucleus ? args.rows_d : 0) + (args.t.nucleus ? args.rows_t : 0);
  if (rows == 0) return cudaSuccess;
  const int64_t narrow = (args.d.nucleus && args.d.V <= kWarpRowMax ? args.rows_d : 0) +
                         (args.t.nucleus && args.t.V <= kWarpRowMax ? args.rows_t : 0);
  if (narrow > 0) {  // narrow rows: one warp each first
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(std::min<int64_t>((narrow + kWWarps - 1) / kWWarps,
                                                  int64_t(sm_count) * 3)));
    cfg.blockDim = dim3(kWWarps * 32);
    cfg.dynamicSmemBytes = kWWarps * sizeof(NucWarpSmem);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, nucleus_warp_kernel, args);
    if (e != cudaSuccess) return e;
  }
  // three CTAs of about 59 KB per SM, each streaming one row at a time
  const int64_t blocks = std::min<int64_t>(rows, int64_t(sm_count) * 3);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(blocks));
  cfg.blockDim = dim3(kNT);
  cfg.dynamicSmemBytes = sizeof(NucSmem);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, nucleus_kernel, args);
}

}  // namespace tt
