// Device helpers shared by the HeadGuard kernels: BF16 conversion, warp
// reductions, the warp-distributed Hadamard-128 butterflies and the group
// quantizer.  Every float operation that decides a stored bit (codes, scale,
// zero, reconstructed values) uses an explicit round-to-nearest intrinsic so
// that the compiler can neither fuse nor reorder it.
#pragma once
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "hg_layout.cuh"

namespace hg {

__device__ __forceinline__ float bf16_to_f32(uint32_t h16) { return __uint_as_float(h16 << 16); }

// Two BF16 packed in a 32-bit word -> two floats (low half first).
__device__ __forceinline__ void bf16x2_to_f32(uint32_t w, float& lo, float& hi) {
  lo = __uint_as_float(w << 16);
  hi = __uint_as_float(w & 0xffff0000u);
}

// fp32 -> BF16 bits, round to nearest even (finite inputs and infinities).
__device__ __forceinline__ uint32_t f32_to_bf16_rn(float f) {
  uint32_t u = __float_as_uint(f);
  if ((u & 0x7fffffffu) > 0x7f800000u) return 0x7fc0u;  // NaN
  u += 0x7fffu + ((u >> 16) & 1u);
  return u >> 16;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// fl32(1/sqrt(128)) -- bit pattern 0x3DB504F3.
__device__ __forceinline__ float hadamard_c() { return __uint_as_float(0x3DB504F3u); }

// Normalised Walsh-Hadamard transform of a 128-vector spread over a warp, lane
// l holding channels 4l..4l+3 (Sylvester order).  Stages h = 1, 2 are inside a
// lane, h = 4..64 pair lane l with lane l ^ (h/4).  Each butterfly maps
// (a, b) = (x[j], x[j+h]) to (a + b, a - b); the 1/sqrt(128) factor is one
// multiply after the last stage.  Self-inverse.
__device__ __forceinline__ void fwht128_warp(float (&x)[4], int lane) {
  const float a0 = __fadd_rn(x[0], x[1]), a1 = __fsub_rn(x[0], x[1]);
  const float a2 = __fadd_rn(x[2], x[3]), a3 = __fsub_rn(x[2], x[3]);
  x[0] = __fadd_rn(a0, a2);
  x[2] = __fsub_rn(a0, a2);
  x[1] = __fadd_rn(a1, a3);
  x[3] = __fsub_rn(a1, a3);
#pragma unroll
  for (int m = 1; m < 32; m <<= 1) {
    const bool upper = (lane & m) != 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float p = __shfl_xor_sync(0xffffffffu, x[i], m);
      x[i] = upper ? __fsub_rn(p, x[i]) : __fadd_rn(x[i], p);
    }
  }
  const float c = hadamard_c();
#pragma unroll
  for (int i = 0; i < 4; ++i) x[i] = __fmul_rn(x[i], c);
}

// Metadata pairs {scale, zero}: two fp32 (8 bytes) or, with the 32-bit
// storage model of Sec. 5.4, two binary16 (4 bytes, scale in the low half).
// A binary16 value is rounded to nearest even and saturates at +-65504; the
// codes are then computed against the stored (rounded) scale and zero, so the
// reconstruction uses exactly what the cache holds.  Since the rounded zero
// can lie above the group minimum and the rounded scale below the true step,
// a quotient may fall outside [0, levels]; the clamp of code_of below covers
// it (only quotients in [0, levels] decide a code, and there its near-tie
// bound holds).
__device__ __forceinline__ float half_sat(float x) {
  return __half2float(__float2half_rn(fminf(fmaxf(x, -65504.0f), 65504.0f)));
}
__device__ __forceinline__ void store_meta(char* base, size_t i, float scale, float zero, bool m16) {
  if (m16) {
    // scale and zero are binary16 values already: the conversion is exact
    *reinterpret_cast<__half2*>(base + i * 4) = __floats2half2_rn(scale, zero);
  } else {
    reinterpret_cast<float2*>(base)[i] = make_float2(scale, zero);
  }
}
__device__ __forceinline__ float2 half2_bits_to_float2(uint32_t w) {
  __half2 h;
  *reinterpret_cast<uint32_t*>(&h) = w;
  return __half22float2(h);
}
__device__ __forceinline__ float2 load_meta(const char* base, size_t i, bool m16) {
  if (m16) return half2_bits_to_float2(__ldg(reinterpret_cast<const uint32_t*>(base) + i));
  return __ldg(reinterpret_cast<const float2*>(base) + i);
}

// code = clamp(rint_even(fl32(d / scale)), 0, levels) computed without a
// division in almost every case.  With r = fl32(1 / scale) and q' = fl32(d r),
// q' = (d / scale)(1 + e1)(1 + e2) with |e1|, |e2| <= 2^-24, and the correctly
// rounded quotient q = fl32(d / scale) is within 2^-24 relative of d / scale,
// so |q' - q| <= 3 * 2^-24 * (d / scale) <= 3e-6 for d / scale <= 16.  When q'
// is farther than 2^-17 from every half-integer, q lies strictly on the same
// side of it and rint(q) == rint(q'); otherwise (a near-tie, about 1.5e-5 of
// the values) the IEEE division decides.  Valid while r is a normal finite
// number (scale >= 2^-125); the caller passes fast = false otherwise.
__device__ __forceinline__ uint32_t code_of(float d, float scale, float r, float levels, bool fast) {
  float rq;
  if (fast) {
    const float q = __fmul_rn(d, r);
    rq = rintf(q);
    if (0.5f - fabsf(__fsub_rn(q, rq)) < 7.62939453125e-6f) rq = rintf(__fdiv_rn(d, scale));
  } else {
    rq = rintf(__fdiv_rn(d, scale));
  }
  rq = fminf(fmaxf(rq, 0.0f), levels);
  return (uint32_t)rq;
}

// Reconstruction fl32(fl32(code * scale) + zero).
__device__ __forceinline__ float dequant1(uint32_t code, float scale, float zero) {
  return __fadd_rn(__fmul_rn((float)code, scale), zero);
}

__device__ __forceinline__ uint4 ldg16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint2 ldg8(const void* p) { return __ldg(reinterpret_cast<const uint2*>(p)); }

}  // namespace hg
