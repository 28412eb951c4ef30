// aq_quant.cuh -- the 8-bit activation quantizer rule (Sec. 4.2.3, symmetric form of
// Eq. 3), shared by the quantizer kernel and the int8-output epilogues.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace aq {

// x / s in IEEE fp32, round half to even, NaN -> 0, clip to [-127, 127].
// Fast path: q = x * fl(1/s) lies within 4u|q| = 2^-22 |q| of fl(x / s) (u = 2^-24;
// the derivation is at quant_fast_bits below); for |q| < 128 that is < 3.1e-5, so unless
// q is within 1e-4 of a half-integer both round to the same integer (and for |q| >= 128
// both clip to the same end).  Near a tie, and for NaN/inf, the exact IEEE quotient
// decides.
__device__ __forceinline__ int8_t quant_one(__half h, float s, float rs) {
  const float x = __half2float(h);
  float q = x * rs;
  const float fr = q - floorf(q);
  if (!(fabsf(fr - 0.5f) > 1e-4f)) q = __fdiv_rn(x, s);
  q = rintf(q);
  if (q != q) q = 0.0f;
  q = fminf(fmaxf(q, -127.0f), 127.0f);
  return static_cast<int8_t>(static_cast<int>(q));
}

// Clip to [-127, 127] keeping NaN (min/max with .NaN propagate it).
__device__ __forceinline__ float clip127_keep_nan(float q) {
  float r;
  asm("max.NaN.f32 %0, %1, 0fC2FE0000;\n\tmin.NaN.f32 %0, %0, 0f42FE0000;" : "=f"(r) : "f"(q));
  return r;
}

// The fast path on the FMA/ALU pipes only (no conversion-unit instructions), for an
// fp16 value already widened to fp32.
// Error bound: with u = 2^-24, fl(1/s) and the product x * fl(1/s) each add a relative
// error of at most u, and fl(x / s) one more, so q = x * fl(1/s) satisfies
// |q - fl(x / s)| <= |q| * (3u + u^2) / (1 - 2u - u^2) < 4u |q| = 2^-22 |q|.
// Test: q is clipped to [-127, 127] (for that range clip-then-round equals
// round-then-clip), and qc * (1 - 2^-22) and qc * (1 + 2^-22), which bracket fl(x / s),
// are rounded half to even with one FMA each by adding 1.5 * 2^23 (exact products, one
// rounding at integer spacing).  Rounding is monotonic, so if both ends give the same
// integer, so does fl(x / s): that integer is the code, in the low byte of `bits`.  The
// ends differ near a half-integer (the caller then applies quant_one), and a NaN fails
// the equality.
__device__ __forceinline__ bool quant_fast_bits(float x, float rs, uint32_t& bits) {
  constexpr float kRound = 12582912.0f;             // 1.5 * 2^23
  constexpr float kUp = 1.0000002384185791015625f;   // 1 + 2^-22
  constexpr float kDown = 0.999999761581420898437f;  // 1 - 2^-22
  const float qc = clip127_keep_nan(x * rs);
  const float hi = __fmaf_rn(qc, kUp, kRound);
  const float lo = __fmaf_rn(qc, kDown, kRound);
  bits = __float_as_uint(hi);
  return hi == lo;
}

// Redoes, with the exact rule, the values of a group of 16 (value i: the half (i & 1) of
// h[i >> 1]) that quant_fast_bits rejects, one value per lane per round: the warp runs
// as many rounds as its busiest lane has rejected values (the selects keep h and qb in
// registers).
__device__ __forceinline__ void quant_fix16(const __half2 (&h)[8], uint32_t (&qb)[16], float s,
                                            float rs) {
  uint32_t slow = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float2 xf = __half22float2(h[i]);
    uint32_t unused;
    slow |= quant_fast_bits(xf.x, rs, unused) ? 0u : 1u << (2 * i);
    slow |= quant_fast_bits(xf.y, rs, unused) ? 0u : 1u << (2 * i + 1);
  }
  while (slow) {
    const int i = __ffs(slow) - 1;
    slow &= slow - 1;
    __half v = __low2half(h[0]);
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (k == i) v = (k & 1) ? __high2half(h[k >> 1]) : __low2half(h[k >> 1]);
    const uint32_t code = static_cast<uint8_t>(quant_one(v, s, rs));
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (k == i) qb[k] = code;
  }
}

// Four codes (low bytes of a, b, c, d) packed into one word, a in the lowest byte.
__device__ __forceinline__ uint32_t pack_low_bytes(uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  return __byte_perm(__byte_perm(a, b, 0x0040), __byte_perm(c, d, 0x0040), 0x5410);
}

}  // namespace aq
