// aq_skinny.cu -- the AQ x A8 linear layer for a few tokens (T <= 16), in one pass.
//
// With few tokens the layer is bound by reading its codes (a few hundred KB), not by
// arithmetic, and every extra launch or partial-sum round trip shows.  Here one CTA
// owns four complete output rows: its threads stride the K/8 group columns, decode
// each group (Eq. 4: fp32 sum of the M codewords, one RNE to fp16) for the four rows
// into registers, multiply with every token's int8 activations on CUDA cores (fp32
// accumulate), and reduce over the CTA in a fixed order (warp butterflies, then the
// warps); the epilogue applies s_x * scale[n] and bias[n] (fp16, fp32, or the next
// layer's int8 activations).  No workspace, no second kernel.
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"
#include "aq_quant.cuh"

namespace aq {

constexpr int kSkinnyRowsPerThread = 4;

// 8 int8 -> 8 floats
__device__ __forceinline__ void i8x8_to_f32(uint2 v, float (&x)[8]) {
  const int32_t a = static_cast<int32_t>(v.x), b = static_cast<int32_t>(v.y);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[i] = static_cast<float>((a << (24 - 8 * i)) >> 24);
    x[4 + i] = static_cast<float>((b << (24 - 8 * i)) >> 24);
  }
}

template <int EB, int TT>
__global__ void __launch_bounds__(256, 2) skinny_kernel(const SkinnyParams p) {
  extern __shared__ float4 skinny_smem4[];
  uint4* sbook = reinterpret_cast<uint4*>(skinny_smem4);                 // [M][256] (8-bit)
  float* wred = reinterpret_cast<float*>(skinny_smem4) + (EB == 1 ? p.M * 256 * 4 : 0);
  grid_dependency_wait();
  allow_dependents();
  const uint4* books = static_cast<const uint4*>(p.books);
  if constexpr (EB == 1) {
    for (int i = threadIdx.x; i < p.M * 256; i += blockDim.x) sbook[i] = books[i];
    __syncthreads();
  }
  // CTA = four output rows; thread = a stride of group columns (8 weights of K each)
  const int n0 = blockIdx.x * kSkinnyRowsPerThread;
  const int G = p.K >> 3;
  const int M = p.M;
  const int T = p.T;
  float acc[kSkinnyRowsPerThread][TT];
#pragma unroll
  for (int r = 0; r < kSkinnyRowsPerThread; ++r)
#pragma unroll
    for (int t = 0; t < TT; ++t) acc[r][t] = 0.0f;

  for (int gi = threadIdx.x; gi < G; gi += blockDim.x) {
    const int kb = gi >> 3, j = gi & 7;
    // the group's decoded weights for the four rows (the decode rule of Eq. 4)
    float w[kSkinnyRowsPerThread][8];
#pragma unroll
    for (int r = 0; r < kSkinnyRowsPerThread; ++r) {
      const int n = n0 + r;
      float s[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) s[e] = 0.0f;
      if (n < p.N) {
        const int64_t cidx = ((static_cast<int64_t>(kb) * p.N + n) * 8 + j) * M;
        for (int m = 0; m < M; ++m) {
          uint4 cw;
          if constexpr (EB == 1) {
            cw = sbook[m * 256 + __ldg(static_cast<const uint8_t*>(p.codes) + cidx + m)];
          } else {
            const int c = __ldg(static_cast<const uint16_t*>(p.codes) + cidx + m);
            cw = __ldg(books + (static_cast<int64_t>(m) << 16) + c);
          }
          const __half2* h2 = reinterpret_cast<const __half2*>(&cw);
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float2 f = __half22float2(h2[i]);
            s[2 * i] = m == 0 ? f.x : __fadd_rn(s[2 * i], f.x);
            s[2 * i + 1] = m == 0 ? f.y : __fadd_rn(s[2 * i + 1], f.y);
          }
        }
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) w[r][e] = __half2float(__float2half_rn(s[e]));
    }
    const int k0 = gi * 8;
#pragma unroll
    for (int t = 0; t < TT; ++t) {
      if (t < T) {
        float x[8];
        i8x8_to_f32(__ldg(reinterpret_cast<const uint2*>(p.xq + static_cast<int64_t>(t) * p.K + k0)), x);
#pragma unroll
        for (int r = 0; r < kSkinnyRowsPerThread; ++r)
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[r][t] = fmaf(w[r][e], x[e], acc[r][t]);
      }
    }
  }
  // reduce over the CTA in a fixed order: butterflies within each warp, then the warps
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kSkinnyRowsPerThread; ++r)
#pragma unroll
    for (int t = 0; t < TT; ++t) {
      float v = acc[r][t];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) wred[(warp * kSkinnyRowsPerThread + r) * TT + t] = v;
    }
  __syncthreads();
  const int nwarps = blockDim.x >> 5;
  const float rs_out = p.out_q8 ? __frcp_rn(p.s_out) : 0.0f;
  for (int o = threadIdx.x; o < kSkinnyRowsPerThread * T; o += blockDim.x) {
    const int t = o / kSkinnyRowsPerThread;
    const int r = o - t * kSkinnyRowsPerThread;
    const int n = n0 + r;
    if (n >= p.N) continue;
    float v = 0.0f;
    for (int wi = 0; wi < nwarps; ++wi) v += wred[(wi * kSkinnyRowsPerThread + r) * TT + t];
    v = fmaf(v, p.s_x * __half2float(p.scale[n]), p.bias ? __half2float(p.bias[n]) : 0.0f);
    const int64_t off = static_cast<int64_t>(t) * p.N + n;
    if (p.out_f32)
      static_cast<float*>(p.y)[off] = v;
    else if (p.out_q8)
      static_cast<int8_t*>(p.y)[off] = quant_one(__float2half_rn(v), p.s_out, rs_out);
    else
      static_cast<__half*>(p.y)[off] = __float2half_rn(v);
  }
}

size_t skinny_smem_bytes(int M, int B, int T, int threads) {
  const int TT = T <= 1 ? 1 : T <= 2 ? 2 : T <= 4 ? 4 : T <= 8 ? 8 : 16;
  return (B == 8 ? static_cast<size_t>(M) * 256 * 16 : 0) +
         static_cast<size_t>(threads / 32) * kSkinnyRowsPerThread * TT * 4;
}

template <int EB>
cudaError_t launch_skinny_eb(const SkinnyParams& p, int blocks, int threads, size_t smem,
                             cudaStream_t st) {
  const dim3 grid(static_cast<unsigned>(blocks)), block(static_cast<unsigned>(threads));
  auto go = [&](auto kernel) -> cudaError_t {
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(smem));
      if (e != cudaSuccess) return e;
    }
    return launch_pdl(kernel, grid, block, smem, st, p);
  };
  if (p.T <= 1) return go(skinny_kernel<EB, 1>);
  if (p.T <= 2) return go(skinny_kernel<EB, 2>);
  if (p.T <= 4) return go(skinny_kernel<EB, 4>);
  if (p.T <= 8) return go(skinny_kernel<EB, 8>);
  return go(skinny_kernel<EB, 16>);
}

cudaError_t launch_skinny(SkinnyParams p, cudaStream_t st) {
  // one CTA per four rows; its threads (a multiple of 32, at most 256) stride the
  // K/8 group columns
  const int G = p.K / 8;
  int threads = (G + 31) / 32 * 32;
  if (threads > 256) threads = 256;
  p.quads = 1;
  const int blocks = (p.N + kSkinnyRowsPerThread - 1) / kSkinnyRowsPerThread;
  const size_t smem = skinny_smem_bytes(p.M, p.B, p.T, threads);
  return p.B == 8 ? launch_skinny_eb<1>(p, blocks, threads, smem, st)
                  : launch_skinny_eb<2>(p, blocks, threads, smem, st);
}

}  // namespace aq
