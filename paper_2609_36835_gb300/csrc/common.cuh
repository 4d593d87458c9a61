// Shared device helpers of the ARC-KV CUDA library (sm_103a).
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <math.h>

#include "arckv.h"

namespace arckv {

typedef __nv_bfloat16 bf16;

// Device status word layout (first 256 bytes of every workspace).
struct DevStatus {
  unsigned int code;       // first arckv_status recorded on the device (0 = OK)
  unsigned int pad[63];
};

__device__ __forceinline__ void set_status(DevStatus* st, unsigned int code) {
  atomicCAS(&st->code, 0u, code);
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(bf16 x) { return __bfloat162float(x); }

// e^x evaluated as 2^(x log2 e): callers fold log2 e into an FMA with their
// shift (e^(x - m) = ex2(x * kLog2e - m * kLog2e)) and take one MUFU ex2
// (relative error ~2^-22; flushes subnormal results to zero).
constexpr float kLog2e = 1.4426950408889634f;
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// bf16x2 triple of two fp32 values (split3_bf16 elementwise, packed pairs).
__device__ __forceinline__ void split3_bf16x2(float a, float b, __nv_bfloat162& h, __nv_bfloat162& m,
                                              __nv_bfloat162& l) {
  h = __floats2bfloat162_rn(a, b);
  const float2 hf = __bfloat1622float2(h);
  const float ea = a - hf.x, eb = b - hf.y;
  m = __floats2bfloat162_rn(ea, eb);
  const float2 mf = __bfloat1622float2(m);
  l = __floats2bfloat162_rn(ea - mf.x, eb - mf.y);
}

// Monotone map of fp32 onto uint32 (total order of finite values).
__device__ __forceinline__ unsigned int f32_ordered(float f) {
  unsigned int u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float f32_from_ordered(unsigned int u) {
  return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}

// bf16 pair (hi, lo) with hi = bf16(x) and lo = bf16(x - hi): x = hi + lo to
// within 2^-16 relative, the operand format of the split tensor-core GEMMs.
__device__ __forceinline__ void split_bf16(float x, bf16& hi, bf16& lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// bf16 triple (h, m, l) with x = h + m + l to within 2^-24 relative: an fp32
// value carried exactly enough for fp32-grade tensor-core products against an
// exact bf16 operand.
__device__ __forceinline__ void split3_bf16(float x, bf16& h, bf16& m, bf16& l) {
  h = __float2bfloat16_rn(x);
  const float r1 = x - __bfloat162float(h);
  m = __float2bfloat16_rn(r1);
  l = __float2bfloat16_rn(r1 - __bfloat162float(m));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Combine two (max, sum of exp(x - max)) pairs.
__device__ __forceinline__ void lse_combine(float& m, float& s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) { m = m2; s = s2; return; }
  if (m2 > m) { s = s * expf(m - m2) + s2; m = m2; }
  else        { s = s + s2 * expf(m2 - m); }
}

inline int cdiv(long long a, long long b) { return (int)((a + b - 1) / b); }

}  // namespace arckv
