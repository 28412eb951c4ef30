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

// The fast path of quant_one alone, for code that quantizes many values at once:
// returns false (and the caller must use quant_one) when x*fl(1/s) lies within 1e-4
// of a half-integer or is not finite.  |q - rint(q)| < 0.4999 is the same test as
// |frac(q) - 1/2| > 1e-4; NaN fails it.  rint rounds half to even, as rintf.
__device__ __forceinline__ bool quant_fast(__half h, float rs, int& out) {
  const float q = __half2float(h) * rs;
  const float r = rintf(q);
  out = max(-127, min(127, static_cast<int>(r)));
  return fabsf(q - r) < 0.4999f;
}

}  // namespace aq
