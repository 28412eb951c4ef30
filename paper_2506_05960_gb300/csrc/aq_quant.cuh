// aq_quant.cuh -- the 8-bit activation quantizer rule (Sec. 4.2.3, symmetric form of
// Eq. 3), shared by the quantizer kernel and the int8-output epilogues.
#pragma once

#include <cstdint>
#include <cuda_fp16.h>

namespace aq {

// x / s in IEEE fp32, round half to even, NaN -> 0, clip to [-127, 127].
// Fast path: q = x * fl(1/s) lies within 3 * 2^-24 * |x/s| of fl(x/s); for
// |x/s| < 128 that is < 2.3e-5, so unless q is within 1e-4 of a half-integer
// both round to the same integer (and for |x/s| >= 128 both clip to the same
// end).  Near a tie, and for NaN/inf, the exact IEEE quotient decides.
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

// The fast path on the FMA/ALU pipes only (no conversion-unit instructions), for an
// fp16 value already widened to fp32: q = x * fl(1/s) is clipped to [-127, 127] first
// (for that range clip-then-round equals round-then-clip) and rounded half to even by
// adding 1.5 * 2^23, which leaves the integer in the low bits of the sum: the low byte
// of `bits` is the int8 code.
// When is rint(q) the rule's rint(fl(x / s))?  With u = 2^-24, fl(1/s) and the product
// each add a relative error of at most u, and fl(x / s) one more, so
// |q - fl(x / s)| <= |q| * (3u + u^2) / (1 - 2u - u^2) < 4u |q|.  If q is farther than
// that from every half-integer, both round to the same integer.  The test
// |q - rint(q)| < 1/2 - 4u |q| is evaluated with an exact subtraction and a threshold
// whose rounding (<= 2^-26) stays below the margin u |q| for |q| >= 1/4; below 1/4 the
// nearest half-integer is more than 1/4 away and the answer is 0 either way.  Returns
// false for a NaN or a value that fails the test: the caller applies quant_one.
__device__ __forceinline__ bool quant_fast_bits(float x, float rs, uint32_t& bits) {
  constexpr float kRound = 12582912.0f;        // 1.5 * 2^23
  constexpr float kFourU = 2.384185791015625e-7f;  // 2^-22
  const float q = x * rs;
  const float qc = fminf(fmaxf(q, -127.0f), 127.0f);
  const float t = __fadd_rn(qc, kRound);
  bits = __float_as_uint(t);
  const float thr = __fmaf_rn(-fabsf(qc), kFourU, 0.5f);
  return fabsf(__fsub_rn(qc, __fsub_rn(t, kRound))) < thr && q == q;
}

// Redoes the values of a group of 16 that quant_fast_bits rejected (bit i of `slow`:
// value i, the half (i & 1) of h[i >> 1]) with the exact rule, one value per lane per
// round: the warp runs as many rounds as its busiest lane has rejected values (the
// selects keep h and qb in registers).
__device__ __forceinline__ void quant_fix16(uint32_t slow, const __half2 (&h)[8],
                                            uint32_t (&qb)[16], float s, float rs) {
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
