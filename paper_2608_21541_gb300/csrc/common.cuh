// common.cuh — shared device helpers of the CertKV library (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

namespace certkv {

constexpr int kD = 128;          // head dimension supported by the kernels
constexpr int kChunk = 128;      // ranks per dispersion chunk (one warp)
constexpr int kHullSeg = 256;    // curve points per hull-filter thread
constexpr int kGroupSegs = 4;    // hull-filter segments per group
constexpr int kSortTile = 2048;  // keys per radix-sort tile
constexpr int kSortThreads = 256;
constexpr uint32_t kFull = 0xffffffffu;

// ------------------------------------------------------------ status word --
// Lives in the first bytes of the workspace; bits are CERTKV_STATUS_*.
__device__ __forceinline__ void raise_status(uint32_t* status, uint32_t bit) {
  atomicOr(status, bit);
}

// ------------------------------------------------------- bounds checks --
// In a library built with -DCERTKV_DEBUG, CERTKV_IN_BOUNDS(cond, status)
// evaluates cond and, when it is false, sets CERTKV_STATUS_BOUNDS (4th bit of
// the status word, if status is not null) and yields false so that the caller
// skips the access; in the normal build it is the constant true and the
// condition is not evaluated.
#ifdef CERTKV_DEBUG
__device__ __forceinline__ bool in_bounds(bool ok, uint32_t* status) {
  if (!ok && status) atomicOr(status, 8u);
  return ok;
}
#define CERTKV_IN_BOUNDS(cond, status) (::certkv::in_bounds((cond), (status)))
#else
#define CERTKV_IN_BOUNDS(cond, status) (true)
#endif

// -------------------------------------------------------------- bf16 ------
__device__ __forceinline__ float bf16lo(uint32_t packed) {
  return __uint_as_float(packed * 65536u);  // the shift by 16 as a multiply (FMA pipe)
}
__device__ __forceinline__ float bf16hi(uint32_t packed) {
  return __uint_as_float(packed & 0xffff0000u);
}

// Round the double-float value hi + lo to bf16, nearest even, in one step:
// hi decides unless it sits exactly half-way, where the sign of lo breaks the tie.
__device__ __forceinline__ uint16_t df_to_bf16(float hi, float lo) {
  uint32_t u = __float_as_uint(hi);
  if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)((u >> 16) | ((u & 0xffffu) ? 0x40u : 0u));
  uint32_t rem = u & 0xffffu;
  uint32_t base = u >> 16;
  bool up;
  if (rem > 0x8000u) up = true;
  else if (rem < 0x8000u) up = false;
  else if (lo != 0.0f) up = ((lo > 0.0f) == (hi > 0.0f));
  else up = (base & 1u) != 0u;
  return (uint16_t)(base + (up ? 1u : 0u));
}

// ----------------------------------------------------- double-float (df) --
// Unevaluated sums hi + lo of two floats (Dekker / Knuth error-free
// transformations); the explicit _rn intrinsics keep the compiler from fusing
// or reassociating the steps.
struct DF {
  float hi, lo;
};

__device__ __forceinline__ DF df_make(float x) { return DF{x, 0.0f}; }

__device__ __forceinline__ DF two_sum(float a, float b) {
  float s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return DF{s, e};
}

__device__ __forceinline__ DF fast_two_sum(float a, float b) {  // |a| >= |b|
  float s = __fadd_rn(a, b);
  float e = __fsub_rn(b, __fsub_rn(s, a));
  return DF{s, e};
}

__device__ __forceinline__ DF two_prod(float a, float b) {
  float p = __fmul_rn(a, b);
  float e = __fmaf_rn(a, b, -p);
  return DF{p, e};
}

__device__ __forceinline__ DF df_add(DF x, DF y) {
  DF s = two_sum(x.hi, y.hi);
  DF t = two_sum(x.lo, y.lo);
  float e = __fadd_rn(s.lo, t.hi);
  DF v = fast_two_sum(s.hi, e);
  e = __fadd_rn(t.lo, v.lo);
  return fast_two_sum(v.hi, e);
}

// x + y for x and y of the same sign (both >= 0 here): the high parts are
// added exactly (two_sum), the low parts folded into the error, one
// renormalisation.  Without cancellation this simplified double-float sum is
// accurate to a few units of 2^-48 (Dekker 1971); it is not used where the
// operands can have opposite signs.
__device__ __forceinline__ DF df_add_same_sign(DF x, DF y) {
  const DF s = two_sum(x.hi, y.hi);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(x.lo, y.lo)));
}

__device__ __forceinline__ DF df_add_f(DF x, float y) {
  DF s = two_sum(x.hi, y);
  float e = __fadd_rn(s.lo, x.lo);
  return fast_two_sum(s.hi, e);
}

__device__ __forceinline__ DF df_neg(DF x) { return DF{-x.hi, -x.lo}; }

__device__ __forceinline__ DF df_mul(DF x, DF y) {
  DF p = two_prod(x.hi, y.hi);
  float e = __fmaf_rn(x.hi, y.lo, p.lo);
  e = __fmaf_rn(x.lo, y.hi, e);
  return fast_two_sum(p.hi, e);
}

__device__ __forceinline__ DF df_mul_f(DF x, float y) {
  DF p = two_prod(x.hi, y);
  float e = __fmaf_rn(x.lo, y, p.lo);
  return fast_two_sum(p.hi, e);
}

// x / y for y != 0: one Newton correction of the float quotient.
__device__ __forceinline__ DF df_div(DF x, DF y) {
  float q1 = __fdiv_rn(x.hi, y.hi);
  DF r = df_add(x, df_neg(df_mul_f(y, q1)));
  float q2 = __fdiv_rn(r.hi, y.hi);
  return fast_two_sum(q1, q2);
}

// sqrt of a non-negative df value: float sqrt plus one Newton correction.
__device__ __forceinline__ DF df_sqrt(DF x) {
  if (!(x.hi > 0.0f)) return DF{0.0f, 0.0f};
  float s = sqrtf(x.hi);
  DF s2 = two_prod(s, s);
  float r = __fadd_rn(__fsub_rn(__fsub_rn(x.hi, s2.hi), s2.lo), x.lo);
  float corr = __fdiv_rn(r, __fmul_rn(2.0f, s));
  return fast_two_sum(s, corr);
}

// sqrt of a non-negative df value from the hardware reciprocal square root:
// s = x * rsqrt(x) is within a few 2^-23 of sqrt(x); one Newton step for the
// square root, s + (x - s^2) / (2 s), with x - s^2 formed exactly (two_prod)
// and 1 / (2 s) taken as rsqrt(x) / 2, squares that error to ~2^-44.
__device__ __forceinline__ DF df_sqrt_newton(DF x) {
  if (!(x.hi > 0.0f)) return DF{0.0f, 0.0f};
  if (x.hi < 7.8886091e-31f) return df_sqrt(x);  // below 2^-100: keep clear of subnormals
  const float r = rsqrtf(x.hi);
  const float s = __fmul_rn(x.hi, r);
  const DF s2 = two_prod(s, s);
  const float e = __fadd_rn(__fsub_rn(__fsub_rn(x.hi, s2.hi), s2.lo), x.lo);
  return fast_two_sum(s, __fmul_rn(e, __fmul_rn(0.5f, r)));
}

__device__ __forceinline__ double df_to_double(DF x) { return (double)x.hi + (double)x.lo; }

__device__ __forceinline__ DF shfl_df(DF x, int src) {
  return DF{__shfl_sync(kFull, x.hi, src), __shfl_sync(kFull, x.lo, src)};
}
__device__ __forceinline__ DF shfl_xor_df(DF x, int m) {
  return DF{__shfl_xor_sync(kFull, x.hi, m), __shfl_xor_sync(kFull, x.lo, m)};
}

__device__ __forceinline__ DF warp_sum_df(DF x) {
#pragma unroll
  for (int m = 16; m >= 1; m >>= 1) x = df_add(x, shfl_xor_df(x, m));
  return x;
}

// Two-wide fp32 arithmetic: one instruction for a pair (sm_100 family).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rc, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " mov.b64 rc, {%6, %7};\n fma.rn.f32x2 rd, ra, rb, rc;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " add.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  float2 d;
  asm("{\n .reg .b64 ra, rb, rd;\n mov.b64 ra, {%2, %3};\n mov.b64 rb, {%4, %5};\n"
      " mul.rn.f32x2 rd, ra, rb;\n mov.b64 {%0, %1}, rd;\n}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

// Monotone 64-bit key of a non-negative df value (for atomicMax).
__device__ __forceinline__ unsigned long long df_order_key(DF x) {
  uint32_t h = __float_as_uint(x.hi);
  uint32_t l = __float_as_uint(x.lo);
  l = (l & 0x80000000u) ? ~l : (l | 0x80000000u);
  return ((unsigned long long)h << 32) | l;
}
__device__ __forceinline__ DF df_from_order_key(unsigned long long k) {
  uint32_t h = (uint32_t)(k >> 32);
  uint32_t l = (uint32_t)k;
  l = (l & 0x80000000u) ? (l & 0x7fffffffu) : ~l;
  return DF{__uint_as_float(h), __uint_as_float(l)};
}

// Sort key of a score: ascending keys = descending non-negative scores.
__device__ __forceinline__ uint32_t score_key(float a) { return ~__float_as_uint(a); }
__device__ __forceinline__ float key_score(uint32_t k) { return __uint_as_float(~k); }

// -------------------------------------------------------------- reductions
__device__ __forceinline__ float warp_max(float x) {
#pragma unroll
  for (int m = 16; m >= 1; m >>= 1) x = fmaxf(x, __shfl_xor_sync(kFull, x, m));
  return x;
}

// Eight per-lane partials of rows 0..7 -> every lane l holds the lane sum of
// row (l & 7).
__device__ __forceinline__ float reduce8(float (&v)[8], int lane) {
#pragma unroll
  for (int o = 4; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float keep = upper ? v[i + o] : v[i];
      const float send = upper ? v[i] : v[i + o];
      v[i] = keep + __shfl_xor_sync(kFull, send, o);
    }
  }
  float x = v[0];
  x += __shfl_xor_sync(kFull, x, 8);
  x += __shfl_xor_sync(kFull, x, 16);
  return x;
}

}  // namespace certkv
