// rowpass.cu -- one streaming pass over logits rows: per row chunk of kChunk
// elements, the maximum m of s_x = z_x * log2(e) / T and the sum of 2^(s_x - m).
//
// These partials are everything the softmax normalisers of Alg. 2 / Alg. 4
// need (log2 sum_x 2^s_x = M + log2 sum_c s_c 2^(m_c - M)), and they double as
// the coarse level of the residual inverse CDF, so every logit is read from HBM
// exactly once. Draft rows that no target position maps to are skipped.
// Target row j < m leaves its scored token t_j out of the sum; the decision
// kernel adds that one term back exactly (no cancellation when the residual
// removes it).
#include <algorithm>
#include <cstdint>

#include "tt_device.cuh"
#include "tt_launch.h"

namespace tt {

namespace {

template <int DT>
struct Vec;
template <>
struct Vec<TT_F32> {
  static constexpr int kElems = 4;
  static constexpr uint32_t kNegInf = 0xff800000u;
};
template <>
struct Vec<TT_BF16> {
  static constexpr int kElems = 8;
  static constexpr uint32_t kNegInf = 0xff80ff80u;  // two bf16 -inf
};

template <int DT>
__device__ __forceinline__ float elem(const uint4& v, int q) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (DT == TT_F32) {
    return __uint_as_float(w[q]);
  } else {
    const uint32_t x = w[q >> 1];
    return __uint_as_float((q & 1) ? (x & 0xffff0000u) : (x << 16));
  }
}

// Replaces element q (0..VEC-1) of a vector by raw bits, with selects only
// (no dynamic register indexing).
template <int DT>
__device__ __forceinline__ void set_elem_bits(uint4& v, int q, uint32_t bits) {
  if constexpr (DT == TT_F32) {
    v.x = q == 0 ? bits : v.x;
    v.y = q == 1 ? bits : v.y;
    v.z = q == 2 ? bits : v.z;
    v.w = q == 3 ? bits : v.w;
  } else {
    const int h = q >> 1;
    const bool high = (q & 1) != 0;
    auto upd = [&](uint32_t x) {
      return high ? ((x & 0x0000ffffu) | (bits << 16)) : ((x & 0xffff0000u) | (bits & 0xffffu));
    };
    v.x = h == 0 ? upd(v.x) : v.x;
    v.y = h == 1 ? upd(v.y) : v.y;
    v.z = h == 2 ? upd(v.z) : v.z;
    v.w = h == 3 ? upd(v.w) : v.w;
  }
}

template <int DT>
__device__ __forceinline__ void process_chunk(const RowSet& S, int64_t r, int c, int excl_col,
                                              float* red_m, float* red_s) {
  constexpr int VEC = Vec<DT>::kElems;
  constexpr int NV = kChunk / (VEC * kRowThreads);
  constexpr int ESZ = DT == TT_F32 ? 4 : 2;
  const int tid = threadIdx.x;
  const char* row = S.data + r * S.stride_bytes;
  const int c0 = c * kChunk;
  const int n = min(kChunk, S.V - c0);

  uint4 buf[NV];
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const int e = (v * kRowThreads + tid) * VEC;
    if (e + VEC <= n) {
      buf[v] = ld_stream_v4(row + size_t(c0 + e) * ESZ);
    } else {
      buf[v] = make_uint4(Vec<DT>::kNegInf, Vec<DT>::kNegInf, Vec<DT>::kNegInf,
                          Vec<DT>::kNegInf);
#pragma unroll
      for (int q = 0; q < VEC; ++q) {  // ragged tail of the row
        if (e + q < n) {
          const uint32_t bits = DT == TT_F32
              ? __ldg(reinterpret_cast<const unsigned int*>(row) + c0 + e + q)
              : uint32_t(__ldg(reinterpret_cast<const unsigned short*>(row) + c0 + e + q));
          set_elem_bits<DT>(buf[v], q, bits);
        }
      }
    }
  }
  const int ex = excl_col - c0;  // the scored token leaves the sum
  if (ex >= 0 && ex < n) {
#pragma unroll
    for (int v = 0; v < NV; ++v) {
      const int e = (v * kRowThreads + tid) * VEC;
      if (ex >= e && ex < e + VEC)
        set_elem_bits<DT>(buf[v], ex - e, DT == TT_F32 ? 0xff800000u : 0xff80u);
    }
  }

  const float scale = S.scale;
  float mx = -INFINITY;
#pragma unroll
  for (int v = 0; v < NV; ++v)
#pragma unroll
    for (int q = 0; q < VEC; ++q) mx = fmaxf(mx, elem<DT>(buf[v], q) * scale);
  float sum = 0.f;
  if (mx != -INFINITY) {
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
      for (int q = 0; q < VEC; ++q) sum += ex2_approx(fmaf(elem<DT>(buf[v], q), scale, -mx));
  }
  warp_merge_ms(mx, sum);
  const int warp = tid >> 5, lane = tid & 31;
  if (lane == 0) {
    red_m[warp] = mx;
    red_s[warp] = sum;
  }
  __syncthreads();
  if (warp == 0) {
    float m2 = lane < kRowThreads / 32 ? red_m[lane] : -INFINITY;
    float s2 = lane < kRowThreads / 32 ? red_s[lane] : 0.f;
    warp_merge_ms(m2, s2);
    if (lane == 0) S.part[r * S.nch + c] = Partial{m2, s2};
  }
}

template <int DTD, int DTT>
__global__ void __launch_bounds__(kRowThreads) rowpass_kernel(RowPassArgs a) {
  __shared__ float red_m[2][kRowThreads / 32];
  __shared__ float red_s[2][kRowThreads / 32];
  const int64_t total = a.items_t + a.items_d;
  int it = 0;
  // target items first: they do not depend on the alignment
  for (int64_t item = blockIdx.x; item < total; item += gridDim.x) {
    if (item < a.items_t) {
      const int64_t r = item / a.t.nch;
      const int c = int(item - r * a.t.nch);
      const int excl = a.excl ? a.excl[r] : -1;
      process_chunk<DTT>(a.t, r, c, excl, red_m[it & 1], red_s[it & 1]);
    } else {
      const int64_t di = item - a.items_t;
      const int64_t r = di / a.d.nch;
      const int c = int(di - r * a.d.nch);
      if (a.d.need && !a.d.need[r]) continue;
      process_chunk<DTD>(a.d, r, c, -1, red_m[it & 1], red_s[it & 1]);
    }
    ++it;
  }
}

template <int DTD, int DTT>
cudaError_t launch_rowpass_t(const RowPassArgs& a, cudaStream_t stream, int sm_count) {
  static int per_sm = 0;
  if (per_sm == 0) {
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &per_sm, rowpass_kernel<DTD, DTT>, kRowThreads, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
  }
  const int64_t total = a.items_t + a.items_d;
  if (total == 0) return cudaSuccess;
  const int64_t grid = std::min<int64_t>(total, int64_t(sm_count) * per_sm);
  rowpass_kernel<DTD, DTT><<<unsigned(grid), kRowThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rowpass(const RowPassArgs& a, int dt_d, int dt_t, cudaStream_t stream,
                           int sm_count) {
  if (dt_d == TT_F32 && dt_t == TT_F32) return launch_rowpass_t<TT_F32, TT_F32>(a, stream, sm_count);
  if (dt_d == TT_F32 && dt_t == TT_BF16) return launch_rowpass_t<TT_F32, TT_BF16>(a, stream, sm_count);
  if (dt_d == TT_BF16 && dt_t == TT_F32) return launch_rowpass_t<TT_BF16, TT_F32>(a, stream, sm_count);
  return launch_rowpass_t<TT_BF16, TT_BF16>(a, stream, sm_count);
}

}  // namespace tt
