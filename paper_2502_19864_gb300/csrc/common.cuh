// common.cuh -- device helpers shared by the libringada kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ra {

typedef __nv_bfloat16 bf16;

// ---- element conversions --------------------------------------------------------------
__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

// ---- reductions ------------------------------------------------------------------------
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

// ---- GELU (sigma of Eq. 1, exact erf form) --------------------------------------------
// erf by Abramowitz & Stegun, Handbook of Mathematical Functions, formula 7.1.28:
//   erf(x) = 1 - (1 + a1 x + ... + a6 x^6)^-16 for x >= 0, odd extension, |error| <= 3e-7.
// Evaluated without cancellation: with e = p - 1 carried exactly through the four squarings
// (p^2k - 1 = e (2 + e)), erf = e16 / (1 + e16); x is clamped at 5, where erf is 1 in fp32.
// Branch-free with one reciprocal; the epilogues that evaluate GELU or GELU' for every
// element of a large tile run it instead of a general-purpose erf.
__device__ __forceinline__ float erf_as7128(float x) {
  const float t = fminf(fabsf(x), 5.0f);
  float p = fmaf(t, 4.30638e-5f, 2.765672e-4f);
  p = fmaf(t, p, 1.520143e-4f);
  p = fmaf(t, p, 9.2705272e-3f);
  p = fmaf(t, p, 4.22820123e-2f);
  float e = __fmul_rn(t, fmaf(t, p, 7.05230784e-2f));  // p - 1
  e = __fmul_rn(e, __fadd_rn(e, 2.0f));  // p^2 - 1
  e = __fmul_rn(e, __fadd_rn(e, 2.0f));  // p^4 - 1
  e = __fmul_rn(e, __fadd_rn(e, 2.0f));  // p^8 - 1
  e = __fmul_rn(e, __fadd_rn(e, 2.0f));  // p^16 - 1
  return copysignf(__fdividef(e, __fadd_rn(e, 1.0f)), x);
}
// GELU(x) = x Phi(x) = h + h erf(x / sqrt 2) with h = x / 2.  The operation sequence (no
// contraction) is the one the packed form below applies to each component, so both give
// bitwise the same result.
__device__ __forceinline__ float gelu_f(float x) {
  const float h = __fmul_rn(x, 0.5f);
  return __fmaf_rn(h, erf_as7128(__fmul_rn(x, 0.70710678118654752f)), h);
}
// d/dx GELU = Phi(x) + x phi(x)
__device__ __forceinline__ float gelu_grad_f(float x) {
  const float Phi = __fmaf_rn(erf_as7128(__fmul_rn(x, 0.70710678118654752f)), 0.5f, 0.5f);
  const float q = __fmul_rn(__fmul_rn(x, -0.5f), x);
  return __fadd_rn(Phi, __fmul_rn(__fmul_rn(x, __expf(q)), 0.39894228040143268f));
}

// ---- packed forms: two values per instruction with the sm_100 fp32x2 arithmetic --------
__device__ __forceinline__ float2 f2(float v) { return make_float2(v, v); }
__device__ __forceinline__ float2 erf2_as7128(float2 x) {
  const float2 t = make_float2(fminf(fabsf(x.x), 5.0f), fminf(fabsf(x.y), 5.0f));
  float2 p = __ffma2_rn(t, f2(4.30638e-5f), f2(2.765672e-4f));
  p = __ffma2_rn(t, p, f2(1.520143e-4f));
  p = __ffma2_rn(t, p, f2(9.2705272e-3f));
  p = __ffma2_rn(t, p, f2(4.22820123e-2f));
  float2 e = __fmul2_rn(t, __ffma2_rn(t, p, f2(7.05230784e-2f)));  // p - 1
  e = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // p^2 - 1
  e = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // p^4 - 1
  e = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // p^8 - 1
  e = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // p^16 - 1
  const float2 d = __fadd2_rn(e, f2(1.0f));
  return make_float2(copysignf(__fdividef(e.x, d.x), x.x), copysignf(__fdividef(e.y, d.y), x.y));
}
__device__ __forceinline__ float2 gelu2(float2 x) {
  const float2 h = __fmul2_rn(x, f2(0.5f));
  return __ffma2_rn(h, erf2_as7128(__fmul2_rn(x, f2(0.70710678118654752f))), h);
}
// GELU(x) and GELU'(x) together (one erf): the same per-component operations as gelu2 and
// gelu_grad2
__device__ __forceinline__ void gelu_both2(float2 x, float2& y, float2& dy) {
  const float2 erf = erf2_as7128(__fmul2_rn(x, f2(0.70710678118654752f)));
  const float2 h = __fmul2_rn(x, f2(0.5f));
  y = __ffma2_rn(h, erf, h);
  const float2 Phi = __ffma2_rn(erf, f2(0.5f), f2(0.5f));
  const float2 q = __fmul2_rn(__fmul2_rn(x, f2(-0.5f)), x);
  const float2 ex = make_float2(__expf(q.x), __expf(q.y));
  dy = __fadd2_rn(Phi, __fmul2_rn(__fmul2_rn(x, ex), f2(0.39894228040143268f)));
}
__device__ __forceinline__ float2 gelu_grad2(float2 x) {
  const float2 Phi = __ffma2_rn(erf2_as7128(__fmul2_rn(x, f2(0.70710678118654752f))), f2(0.5f), f2(0.5f));
  const float2 q = __fmul2_rn(__fmul2_rn(x, f2(-0.5f)), x);
  const float2 ex = make_float2(__expf(q.x), __expf(q.y));
  return __fadd2_rn(Phi, __fmul2_rn(__fmul2_rn(x, ex), f2(0.39894228040143268f)));
}
// 2^x on the special function unit (ex2.approx): about 2 ulp, results below 2^-126 flushed to
// zero -- the softmax probabilities it serves are rounded to bf16, and one below 2^-126
// contributes nothing
__device__ __forceinline__ float ex2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// SiLU and its derivative with the special-function exponential and the fast division (a few
// ulp; they run per element in the SwiGLU epilogues).  For x below about -88 the denominator
// overflows and the sigmoid is 0, its limit.
__device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.0f + __expf(-x)); }
__device__ __forceinline__ float silu_grad_f(float x) {
  const float s = __fdividef(1.0f, 1.0f + __expf(-x));
  return s * (1.0f + x * (1.0f - s));
}

// ---- RoPE ---------------------------------------------------------------------------------
// inverse frequency of rotate-half pair i of a head of dh dims: theta^(-2 i / dh); the angle
// at position s is s times this (every RoPE kernel evaluates it this way)
__device__ __forceinline__ float rope_freq(int i, int dh, float theta) {
  return expf(-logf(theta) * (2.0f * (float)i / (float)dh));
}

// ---- programmatic dependent launch ----------------------------------------------------
// A kernel started with launch_pdl may begin while the kernel before it in the stream is
// still finishing.  pdl_wait() blocks until that kernel has completed and its writes are
// visible; it precedes every access to memory that earlier kernels write or read.
// pdl_trigger() lets the next kernel of the stream be scheduled (its CTAs then wait in their
// own pdl_wait).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---- error word written by kernels whose bounded waits ran out -------------------------
// Bit 0: a wait timed out.  The host reads and clears it in ra_sync_status.
enum : unsigned { RA_DEVERR_TIMEOUT = 1u, RA_DEVERR_BOUNDS = 2u };

__device__ __forceinline__ void set_dev_error(unsigned* flag, unsigned bits) {
  if (flag) atomicOr(flag, bits);
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Upper bound for any single in-kernel wait: far above the longest legitimate wait
// (one tile's main loop, microseconds), short enough that a broken pipeline ends.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

}  // namespace ra
