// tt_device.cuh -- device helpers and the workspace layout shared by the
// kernels of the TokenTiming verification path (sm_103a).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "tt.h"

namespace tt {

constexpr int kChunk = 2048;         // logits columns per row chunk (one partial)
constexpr int kRowThreads = 256;     // threads of the row-pass and decision blocks
constexpr int32_t kInf = 0x3fffffff; // "infinite" accumulated DTW cost

// -------------------------------------------------------------- workspace

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }
__host__ __device__ inline int n_chunks(int V) { return V <= 0 ? 0 : (V + kChunk - 1) / kChunk; }

// Partial of one row chunk: m = max of s_x = z_x * log2(e) / T over the chunk,
// s = sum of 2^(s_x - m) over the chunk (target rows leave out their scored
// token, whose term is rebuilt exactly by the decision kernel).
struct Partial {
  float m;
  float s;
};

// A top-k candidate of a filtered row: the raw logit and its column; a row
// unit's list holds its k best in order (larger logit first, then smaller
// column), padded with (-inf, -1) when the unit has fewer than k columns.
struct Cand {
  float v;
  int32_t c;
};

// Entries between the starts of two consecutive top-k lists: k rounded up to
// an even count, so that every list starts on a 16-byte boundary.
__host__ __device__ inline int cand_stride(int k) { return k + (k & 1); }

// Header of a filtered row's kept set: natural log of the kept normaliser and
// the kept count (0: not finite). A top-k row's set itself is k Cand entries
// holding (probability, column), larger logit first, unused entries (0, -1).
// A nucleus row (top-p without top-k) keeps every column ranked at or before
// (tau, tau_col) in the order larger logit first, then smaller column; its
// kept probabilities are 2^(z * scale - M) * inv_s, and its per-chunk kept
// masses sit in the workspace's um arrays.
struct KeptHead {
  float lse;
  int32_t n;
  float tau;       // nucleus rows: raw logit of the last kept column
  int32_t tau_col; // and that column
  float M;         // nucleus rows: the row's largest z * scale
  float inv_s;     // 1 / (sum over kept columns of 2^(z * scale - M))
};

// A column of a request's repetition-penalty set (its history and sequence
// tokens): the column and the first sequence position holding it (-1 when the
// history holds it), so that a row at position j penalizes it when first < j.
// A request's entries are sorted by column, one per column.
struct PenEntry {
  int32_t col;
  int32_t first;
};

// Sizes of the repetition-penalty arrays of a call (zeros: no penalty).
struct PenSizes {
  int n_hist_d = 0, n_hist_t = 0;  // history entries of each family
  bool on_d = false, on_t = false; // families with a penalty
};

// The row pass hands out work from kWorkShards counters, each on its own
// 256-byte line, so that no single L2 address serialises every CTA's draws.
constexpr int kWorkShards = 8;
constexpr int kWorkStride = 32;  // in 8-byte words

struct Workspace {
  Partial* part_d;   // [n_draft * nch_d]
  Partial* part_t;   // [(n_target + B) * nch_t]
  uint8_t* need_d;   // [n_draft]: draft row is mapped by some target position
  int32_t* map;      // [n_target] alignment map when the caller keeps none
  float* q_hat;      // [n_target] transferred probabilities when the caller keeps none
  int32_t* status;   // [B] per-request status between kernels
  int32_t* excl;     // [n_target + B] scored column of each target row (-1: bonus row)
  int32_t* err;      // two words: epoch of a call whose row pass failed, and why
  unsigned long long* work;  // row-pass work counters (kWorkShards, kWorkStride apart), zeroed
                             // by the kernel before the row pass
  Cand* cand_d;      // [n_draft * nch_d * cand_stride(k_d)] top-k lists of filtered draft rows
  Cand* cand_t;      // [(n_target + B) * nch_t * cand_stride(k_t)] top-k lists of filtered target rows
  Cand* kept_d;      // [n_draft * k_d] kept sets (probability, column) of filtered draft rows
  Cand* kept_t;      // [(n_target + B) * k_t] kept sets of filtered target rows
  KeptHead* head_d;  // [n_draft] their headers
  KeptHead* head_t;  // [n_target + B]
  float* um_d;       // [n_draft * nch_d] kept probability mass per chunk of nucleus draft rows
  float* um_t;       // [(n_target + B) * nch_t] the same for nucleus target rows
  // repetition penalty, per penalized family: each request's sorted penalized
  // columns (at base[b], cnt[b] entries, capacity its history plus its tokens)
  // and, per row unit u, the first entry at or past the unit's first column
  PenEntry* pen_d;    // [n_hist_d + n_draft]
  int32_t* pbase_d;   // [B]
  int32_t* pcnt_d;    // [B]
  int32_t* pstart_d;  // [B * (nch_d + 1)]
  PenEntry* pen_t;    // [n_hist_t + n_target]
  int32_t* pbase_t;   // [B]
  int32_t* pcnt_t;    // [B]
  int32_t* pstart_t;  // [B * (nch_t + 1)]
  int32_t* pstatus;   // [B] problems of the histories (TT_REQ_* bits)
  size_t bytes;
};

// Workspace of a call: k_d / k_t > 0 for families with top-k lists, nuc_d /
// nuc_t for nucleus families (top-p without top-k).
__host__ __device__ inline Workspace workspace_layout(void* base, int B, int n_draft, int n_target,
                                                      int V_d, int V_t, int k_d = 0,
                                                      int k_t = 0, bool nuc_d = false,
                                                      bool nuc_t = false,
                                                      PenSizes pen = PenSizes()) {
  Workspace w;
  char* p = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t n) {
    char* r = p ? p + off : nullptr;
    off = align256(off + n);
    return r;
  };
  const size_t rows_t = size_t(n_target) + B;
  w.part_d = reinterpret_cast<Partial*>(take(sizeof(Partial) * size_t(n_draft) * n_chunks(V_d)));
  w.part_t = reinterpret_cast<Partial*>(take(sizeof(Partial) * rows_t * n_chunks(V_t)));
  w.need_d = reinterpret_cast<uint8_t*>(take(size_t(n_draft)));
  w.map = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * size_t(n_target)));
  w.q_hat = reinterpret_cast<float*>(take(sizeof(float) * size_t(n_target)));
  w.status = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * size_t(B)));
  w.excl = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * rows_t));
  w.err = reinterpret_cast<int32_t*>(take(2 * sizeof(int32_t)));
  w.work = reinterpret_cast<unsigned long long*>(take(kWorkShards * kWorkStride * sizeof(unsigned long long)));
  w.cand_d = reinterpret_cast<Cand*>(
      take(sizeof(Cand) * size_t(n_draft) * n_chunks(V_d) * size_t(k_d > 0 ? cand_stride(k_d) : 0)));
  w.cand_t = reinterpret_cast<Cand*>(
      take(sizeof(Cand) * rows_t * n_chunks(V_t) * size_t(k_t > 0 ? cand_stride(k_t) : 0)));
  w.kept_d = reinterpret_cast<Cand*>(take(sizeof(Cand) * size_t(n_draft) * size_t(k_d > 0 ? k_d : 0)));
  w.kept_t = reinterpret_cast<Cand*>(take(sizeof(Cand) * rows_t * size_t(k_t > 0 ? k_t : 0)));
  const bool hd = k_d > 0 || nuc_d, ht = k_t > 0 || nuc_t;
  w.head_d = reinterpret_cast<KeptHead*>(take(hd ? sizeof(KeptHead) * size_t(n_draft) : 0));
  w.head_t = reinterpret_cast<KeptHead*>(take(ht ? sizeof(KeptHead) * rows_t : 0));
  w.um_d = reinterpret_cast<float*>(take(nuc_d ? sizeof(float) * size_t(n_draft) * n_chunks(V_d) : 0));
  w.um_t = reinterpret_cast<float*>(take(nuc_t ? sizeof(float) * rows_t * n_chunks(V_t) : 0));
  const size_t pd = pen.on_d ? 1 : 0, pt = pen.on_t ? 1 : 0;
  w.pen_d = reinterpret_cast<PenEntry*>(
      take(pd * sizeof(PenEntry) * (size_t(pen.n_hist_d) + size_t(n_draft))));
  w.pbase_d = reinterpret_cast<int32_t*>(take(pd * sizeof(int32_t) * size_t(B)));
  w.pcnt_d = reinterpret_cast<int32_t*>(take(pd * sizeof(int32_t) * size_t(B)));
  w.pstart_d = reinterpret_cast<int32_t*>(
      take(pd * sizeof(int32_t) * size_t(B) * size_t(n_chunks(V_d) + 1)));
  w.pen_t = reinterpret_cast<PenEntry*>(
      take(pt * sizeof(PenEntry) * (size_t(pen.n_hist_t) + size_t(n_target))));
  w.pbase_t = reinterpret_cast<int32_t*>(take(pt * sizeof(int32_t) * size_t(B)));
  w.pcnt_t = reinterpret_cast<int32_t*>(take(pt * sizeof(int32_t) * size_t(B)));
  w.pstart_t = reinterpret_cast<int32_t*>(
      take(pt * sizeof(int32_t) * size_t(B) * size_t(n_chunks(V_t) + 1)));
  w.pstatus = reinterpret_cast<int32_t*>(take((pd | pt) * sizeof(int32_t) * size_t(B)));
  w.bytes = off;
  return w;
}

// ------------------------------------------------------------------ loads

__device__ __forceinline__ float bf16_to_f32(uint16_t h) {
  return __uint_as_float(uint32_t(h) << 16);
}

template <int DT>
__device__ __forceinline__ float load_logit(const void* row, int64_t x) {
  if constexpr (DT == TT_F32) {
    return __ldg(static_cast<const float*>(row) + x);
  } else {
    return bf16_to_f32(__ldg(static_cast<const unsigned short*>(row) + x));
  }
}

// 16-byte streaming load that does not allocate in L1.
__device__ __forceinline__ uint4 ld_stream_v4(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// -------------------------------------------------------------- reductions

// Merge two (max, sum-of-2^(s - max)) pairs.
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2) {
  if (m2 > m) {
    s = s2 + (m == -INFINITY ? 0.f : s * ex2_approx(m - m2));
    m = m2;
  } else if (m2 != -INFINITY) {
    s += s2 * ex2_approx(m2 - m);
  }
}

__device__ __forceinline__ void warp_merge_ms(float& m, float& s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    merge_ms(m, s, m2, s2);
  }
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Log2-normaliser of a row from its chunk partials, computed by one warp:
// returns (M, S) with sum over the row of 2^(s_x - M) = S (excluding what the
// partials exclude). S accumulates in fp64. Rows of up to 128 chunks are read
// once (four partials per lane held in registers).
__device__ __forceinline__ void row_norm_warp(const Partial* part, int nch, int lane, float& M,
                                              double& S) {
  float mx = -INFINITY;
  double acc = 0.0;
  if (nch <= 128) {
    Partial p[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int c = lane + 32 * r;
      p[r] = c < nch ? part[c] : Partial{-INFINITY, 0.f};
      mx = fmaxf(mx, p[r].m);
    }
    mx = warp_max_f(mx);
    if (mx != -INFINITY) {
#pragma unroll
      for (int r = 0; r < 4; ++r)
        if (p[r].m != -INFINITY) acc += double(p[r].s) * double(ex2_approx(p[r].m - mx));
    }
  } else {
    for (int c = lane; c < nch; c += 32) mx = fmaxf(mx, part[c].m);
    mx = warp_max_f(mx);
    if (mx != -INFINITY) {
      for (int c = lane; c < nch; c += 32) {
        const Partial q = part[c];
        if (q.m != -INFINITY) acc += double(q.s) * double(ex2_approx(q.m - mx));
      }
    }
  }
  M = mx;
  S = warp_sum_d(acc);
}

__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 2^y for an fp64 exponent: the split y = n + f (n integer, |f| <= 1/2) is
// exact, 2^f comes from the SFU (relative error about 2^-22) and 2^n is built
// from its exponent bits. Below 2^-1020 the result is 0.
__device__ __forceinline__ double exp2_split(double y) {
  if (!(y > -1020.0)) return 0.0;
  const double n = rint(y);
  const int ni = int(n);
  const double scale = __hiloint2double((ni + 1023) << 20, 0);
  return double(ex2_approx(float(y - n))) * scale;
}

// log2 of a positive fp64 value: exponent exactly, mantissa from the SFU.
__device__ __forceinline__ double log2_split(double v) {
  int e;
  const double m = frexp(v, &e);  // v = m * 2^e, m in [1/2, 1)
  return double(e) + double(lg2_approx(float(m)));
}

// ----------------------------------------------------------------- Philox

__device__ __forceinline__ void philox4x64_10(uint64_t c[4], uint64_t k0, uint64_t k1) {
  const uint64_t M0 = 0xD2E7470EE14C6C93ULL, M1 = 0xCA5A826395121157ULL;
  const uint64_t W0 = 0x9E3779B97F4A7C15ULL, W1 = 0xBB67AE8584CAA73BULL;
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    uint64_t lo0 = M0 * c[0], hi0 = __umul64hi(M0, c[0]);
    uint64_t lo1 = M1 * c[2], hi1 = __umul64hi(M1, c[2]);
    uint64_t n0 = hi1 ^ c[1] ^ k0, n2 = hi0 ^ c[3] ^ k1;
    c[0] = n0;
    c[1] = lo1;
    c[2] = n2;
    c[3] = lo0;
    k0 += W0;
    k1 += W1;
  }
}

// u in [0,1): top 24 bits of word 0 of Philox4x64-10 at counter
// (pos, stream, request, 0), key (seed, 0). Exact in fp32 and fp64.
__device__ __forceinline__ double philox_uniform(uint64_t seed, uint64_t pos, uint64_t stream,
                                                 uint64_t request) {
  uint64_t c[4] = {pos, stream, request, 0};
  philox4x64_10(c, seed, 0);
  return double(c[0] >> 40) * (1.0 / 16777216.0);
}

// Records a failure of call `epoch` (TT_REQ_TIMEOUT / TT_REQ_INTERNAL bits).
// Error report of a call: err[0] = the reporting call's epoch, err[1] = its
// TT_REQ_* bits, updated together as one 64-bit word, so that a report of a
// new call replaces an earlier call's bits instead of adding to them (the
// words never need clearing). The compare-and-swap retries only while other
// reporters of the same call change the word.
__device__ __forceinline__ void report_error(int32_t* err, int32_t epoch, int32_t bits) {
  if (!err) return;
  unsigned long long* w = reinterpret_cast<unsigned long long*>(err);
  unsigned long long seen = __ldcg(w), want;
  do {
    want = seen;
    const uint32_t old_bits = int32_t(uint32_t(want)) == epoch ? uint32_t(want >> 32) : 0u;
    seen = atomicCAS(w, want,
                     (uint64_t(old_bits | uint32_t(bits)) << 32) | uint64_t(uint32_t(epoch)));
  } while (seen != want);
}

// ------------------------------------------------------------ warp sorting

// Bitonic sort of one value per lane across the warp: largest at lane 0
// (DESC) or smallest at lane 0.
template <bool DESC>
__device__ __forceinline__ float warp_sort(float x, int lane) {
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      const float o = __shfl_xor_sync(0xffffffffu, x, j);
      // lanes [i, i + k) form a run sorted descending when (i & k) == 0 (k = 32:
      // the whole warp); the lower lane of a pair keeps the larger value there
      const bool up = ((lane & j) == 0) == (k == 32 || (lane & k) == 0);
      x = (DESC ? up : !up) ? fmaxf(x, o) : fminf(x, o);
    }
  }
  return x;
}

// Sorts a bitonic sequence held one value per lane, largest at lane 0.
__device__ __forceinline__ float warp_merge_desc(float x, int lane) {
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const float o = __shfl_xor_sync(0xffffffffu, x, j);
    x = (lane & j) == 0 ? fmaxf(x, o) : fminf(x, o);
  }
  return x;
}

// ------------------------------------------------------------ CSR helpers

// Offsets of request b are usable: 0 <= off[b] <= off[b+1] <= n.
__device__ __forceinline__ bool csr_ok(const int32_t* off, int b, int n) {
  int a = off[b], e = off[b + 1];
  return a >= 0 && a <= e && e <= n;
}

}  // namespace tt
