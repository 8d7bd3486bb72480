// tt_f2.cuh -- compensated fp32 pairs (an unevaluated sum hi + lo, about
// 2^-44 relative), 2^y with an exact exponent split, and the grid-dependency
// wait, shared by the decision kernels (decide.cu, filter.cu).
#pragma once

#include "tt_device.cuh"

namespace tt {

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

// a * b as a normalised pair.
__device__ __forceinline__ F2 f2_mul_f(F2 a, float b) {
  const float p = __fmul_rn(a.hi, b);
  const float e = fmaf(a.hi, b, -p);
  const float lo = fmaf(a.lo, b, e);
  const float hi = __fadd_rn(p, lo);
  return {hi, __fsub_rn(lo, __fsub_rn(hi, p))};
}

__device__ __forceinline__ bool f2_lt(F2 a, F2 b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}

__device__ __forceinline__ F2 shfl_up_f2(F2 v, int o, int width = 32) {
  return {__shfl_up_sync(0xffffffffu, v.hi, o, width), __shfl_up_sync(0xffffffffu, v.lo, o, width)};
}

// 2^(z * scale - M) with the exponent split exactly (TwoProd, TwoSum, rint);
// only 2^f, |f| <= 1/2, comes from the SFU.
__device__ __forceinline__ float exp2_scaled(float z, float scale, float M) {
  const float xh = __fmul_rn(z, scale);
  const float xl = fmaf(z, scale, -xh);
  const F2 d = two_sum(xh, -M);
  const float n = rintf(d.hi);
  const float f = __fadd_rn(__fsub_rn(d.hi, n), __fadd_rn(d.lo, xl));
  if (!(n > -126.f)) return 0.f;
  return ex2_approx(f) * __int_as_float((int(n) + 127) << 23);
}

__device__ __forceinline__ void grid_dependency_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

}  // namespace tt
