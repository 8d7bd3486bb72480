// pen.cu -- the per-request sets of the repetition penalty (the generation
// hyperparameter table, App. F: 1.1 for the Qwen2.5-0.5B model).
//
// A row's penalized columns are its request's history and the sequence tokens
// before the row's position (target row j: t_1..t_j; draft row i: d_1..d_i).
// pen_prep_kernel (one CTA per request) sorts the request's history and
// sequence columns together, keeps one entry per column with the first
// sequence position holding it (-1 when the history does), so that row j
// penalizes the entry when first < j, and records where each row unit's
// columns start in the sorted entries. The row pass then leaves these columns
// out of its unit lists, and the kept-set kernel adds them back, each with
// the row's own value.
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

constexpr int kPT = 256;
constexpr int kSortCap = 4096;  // history (<= TT_MAX_HISTORY) plus sequence (<= TT_MAX_M)
static_assert(TT_MAX_HISTORY + TT_MAX_M <= kSortCap, "a request's entries fit the sort buffer");

__device__ __forceinline__ bool csr_range(const int32_t* off, int b, int n, int& lo, int& hi) {
  lo = hi = 0;
  if (!off) return true;
  const int a0 = off[b], a1 = off[b + 1];
  if (a0 < 0 || a1 < a0 || a1 > n) return false;
  lo = a0;
  hi = a1;
  return true;
}

__global__ void __launch_bounds__(kPT) pen_prep_kernel(PenArgs a) {
  __shared__ unsigned long long key[kSortCap];
  __shared__ int wsum[kPT / 32];
  __shared__ int s_bad;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int st = 0;
  for (int fam = 0; fam < 2; ++fam) {
    const bool tgt = fam == 1;
    if (!(tgt ? a.on_t : a.on_d)) continue;
    const int V = tgt ? a.V_t : a.V_d;
    int h0, h1, s0, s1;
    if (!csr_range(tgt ? a.hist_off_t : a.hist_off_d, b, tgt ? a.n_hist_t : a.n_hist_d, h0, h1)) {
      st |= TT_REQ_BAD_OFFSETS;
      h0 = h1 = 0;
    }
    if (!csr_range(tgt ? a.target_off : a.draft_off, b, tgt ? a.n_target : a.n_draft, s0, s1))
      s0 = s1 = 0;  // (reported by the other kernels)
    if (h1 - h0 > TT_MAX_HISTORY) {
      st |= TT_REQ_TOO_LONG;
      h1 = h0;
    }
    if (s1 - s0 > TT_MAX_M) s1 = s0;  // (too long: reported by the other kernels)
    const int nh = h1 - h0, ns = s1 - s0, n = nh + ns;
    int N = 1;
    while (N < n) N <<= 1;
    const int32_t* hcols = tgt ? a.hist_cols_t : a.hist_cols_d;
    const int32_t* scols = tgt ? a.target_cols : a.draft_cols;
    if (tid == 0) s_bad = 0;
    __syncthreads();
    // keys (column, first position + 1): history entries first (position -1)
    for (int i = tid; i < N; i += kPT) {
      unsigned long long k = ~0ull;
      if (i < nh) {
        const int c = hcols[h0 + i];
        if (c >= 0 && c < V) k = (static_cast<unsigned long long>(c) << 32);
        else s_bad = 1;
      } else if (i < n) {
        const int c = scols[s0 + (i - nh)];
        if (c >= 0 && c < V) k = (static_cast<unsigned long long>(c) << 32) | unsigned(i - nh + 1);
      }
      key[i] = k;
    }
    __syncthreads();
    if (s_bad) st |= TT_REQ_ID_OUT_OF_RANGE;
    // bitonic sort, ascending
    for (int size = 2; size <= N; size <<= 1)
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        for (int i = tid; i < N / 2; i += kPT) {
          const int lo = 2 * i - (i & (stride - 1));
          const int hi = lo + stride;
          const bool up = (lo & size) == 0;
          const unsigned long long x = key[lo], y = key[hi];
          if ((x > y) == up) {
            key[lo] = y;
            key[hi] = x;
          }
        }
        __syncthreads();
      }
    // one entry per column: the first of its run (smallest position)
    constexpr int kPer = kSortCap / kPT;
    unsigned long long mine[kPer];
    int flags = 0, cnt = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int i = tid * kPer + q;
      mine[q] = i < N ? key[i] : ~0ull;
      const bool f = i < N && mine[q] != ~0ull &&
                     (i == 0 || (key[i - 1] >> 32) != (mine[q] >> 32));
      flags |= int(f) << q;
      cnt += f;
    }
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int base_w = 0, total = 0;
#pragma unroll
    for (int w = 0; w < kPT / 32; ++w) {
      if (w < warp) base_w += wsum[w];
      total += wsum[w];
    }
    const int base = h0 + s0;  // the request's segment (capacity nh + ns >= total)
    PenEntry* out = (tgt ? a.pen_t : a.pen_d) + base;
    int32_t* ucol = reinterpret_cast<int32_t*>(key);  // the sorted unique columns
    __syncthreads();  // every key is read
    int idx = base_w + incl - cnt;
#pragma unroll
    for (int q = 0; q < kPer; ++q)
      if (flags >> q & 1) {
        const int c = int(mine[q] >> 32), first = int(uint32_t(mine[q])) - 1;
        out[idx] = PenEntry{c, first};
        ucol[idx] = c;
        ++idx;
      }
    __syncthreads();
    // the first entry of each row unit (and the count after the last unit)
    const int nlist = tgt ? a.nlist_t : a.nlist_d, unit = tgt ? a.unit_t : a.unit_d;
    const int nch = tgt ? a.nch_t : a.nch_d;
    int32_t* start = (tgt ? a.pstart_t : a.pstart_d) + int64_t(b) * (nch + 1);
    for (int u = tid; u <= nlist; u += kPT) {
      const int64_t c0 = int64_t(u) * unit;
      int lo = 0, hi = total;
      while (lo < hi) {  // first entry with column >= c0
        const int mid = (lo + hi) >> 1;
        if (ucol[mid] < c0) lo = mid + 1;
        else hi = mid;
      }
      start[u] = u == nlist ? total : lo;
    }
    if (tid == 0) {
      (tgt ? a.pbase_t : a.pbase_d)[b] = base;
      (tgt ? a.pcnt_t : a.pcnt_d)[b] = total;
    }
    __syncthreads();  // the buffers are reused by the next family
  }
  if (tid == 0) a.pstatus[b] = st;
}

}  // namespace

cudaError_t preload_pen() {
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, pen_prep_kernel);
}

cudaError_t launch_pen_prep(const PenArgs& args, cudaStream_t stream) {
  if (args.B == 0 || !(args.on_d || args.on_t)) return cudaSuccess;
  pen_prep_kernel<<<args.B, kPT, 0, stream>>>(args);
  return cudaGetLastError();
}

}  // namespace tt
