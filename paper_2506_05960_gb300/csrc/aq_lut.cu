// aq_lut.cu -- lookup-table order of the AQ x A8 layer for small token counts
// (App. A.1, Eq. A5 -> A6, restated for a linear layer):
//   L[t][i][m][c] = sum_{e<g} x[t][g*i + e] * C^(m)[c][e]     for every codeword c
//   acc[t][n]     = sum_i sum_m L[t][i][m][ b[n][i][m] ]
// The weight matrix is never decoded: each output row costs M table reads per
// group instead of g multiply-adds, and the tables cost 2*g*M*2^B flops per
// group and token.  Only 8-bit codes (256-row codebooks) are supported.
//
// One CTA owns a chunk of J consecutive groups (inside one packed 64-wide K
// block) and a slice of output rows: it stages the chunk's int8 activations,
// builds the chunk's tables for all tokens in shared memory, then each thread
// walks its rows, reads the rows' codes with one contiguous load and
// gather-sums the table entries of all tokens (Tp floats per entry, 16-byte
// shared loads).  Chunk partial sums go to the workspace [chunks][T][N] and
// the split reduction applies scale and bias.
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"

namespace aq {

__global__ void __launch_bounds__(256) lut_kernel(const LutParams p) {
  extern __shared__ float4 lut_smem4[];
  float* L = reinterpret_cast<float*>(lut_smem4);              // [J][M][256][Tp]
  const int J = p.J, M = p.M, Tp = p.Tp, T = p.T;
  float* xs = L + static_cast<size_t>(J) * M * 256 * Tp;       // [T][J*8]
  grid_dependency_wait();
  allow_dependents();
  const int chunk = blockIdx.x;
  const int g0 = chunk * J;
  const int nj = min(J, p.G - g0);
  const int kb = g0 >> 3;
  const int jj0 = g0 & 7;

  // stage the chunk's activations as floats (int8 values are exact)
  const int width = J * 8;
  for (int i = threadIdx.x; i < T * width; i += blockDim.x) {
    const int t = i / width;
    const int e = i - t * width;
    xs[i] = (e < nj * 8) ? static_cast<float>(p.xq[static_cast<int64_t>(t) * p.K + g0 * 8 + e])
                         : 0.0f;
  }
  __syncthreads();

  // build: one table entry (group j, codebook m, codeword c) per thread and step
  const int entries = J * M * 256;
  for (int ent = threadIdx.x; ent < entries; ent += blockDim.x) {
    const int j = ent / (M * 256);
    const int r = ent - j * (M * 256);          // m * 256 + c
    const uint4 raw = reinterpret_cast<const uint4*>(p.books)[r];
    const __half2* h2 = reinterpret_cast<const __half2*>(&raw);
    float cw[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __half22float2(h2[i]);
      cw[2 * i] = f.x;
      cw[2 * i + 1] = f.y;
    }
    float4* dst = reinterpret_cast<float4*>(L + static_cast<size_t>(ent) * Tp);
    for (int t4 = 0; t4 < Tp; t4 += 4) {
      float o[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int t = t4 + u;
        float s = 0.0f;
        if (t < T) {
          const float* xr = xs + t * width + j * 8;
#pragma unroll
          for (int e = 0; e < 8; ++e) s = fmaf(xr[e], cw[e], s);
        }
        o[u] = s;
      }
      dst[t4 >> 2] = make_float4(o[0], o[1], o[2], o[3]);
    }
  }
  __syncthreads();

  // gather-sum: one output row per thread and step
  const int n_begin = blockIdx.y * p.rows_per_cta;
  const int n_end = min(p.N, n_begin + p.rows_per_cta);
  const int code_bytes = M;  // 8-bit codes
  for (int n = n_begin + threadIdx.x; n < n_end; n += blockDim.x) {
    float acc[16];
#pragma unroll
    for (int t = 0; t < 16; ++t) acc[t] = 0.0f;
    const uint8_t* codes =
        p.packed + ((static_cast<int64_t>(kb) * p.N + n) * 8 + jj0) * code_bytes;
    for (int j = 0; j < nj; ++j) {
      for (int m = 0; m < M; ++m) {
        const int c = codes[j * M + m];
        const float4* e = reinterpret_cast<const float4*>(L + ((j * M + m) * 256 + c) * Tp);
        const float4 v0 = e[0];
        acc[0] += v0.x; acc[1] += v0.y; acc[2] += v0.z; acc[3] += v0.w;
        if (Tp > 4) {
          const float4 v1 = e[1];
          acc[4] += v1.x; acc[5] += v1.y; acc[6] += v1.z; acc[7] += v1.w;
        }
        if (Tp > 8) {
          const float4 v2 = e[2];
          const float4 v3 = e[3];
          acc[8] += v2.x; acc[9] += v2.y; acc[10] += v2.z; acc[11] += v2.w;
          acc[12] += v3.x; acc[13] += v3.y; acc[14] += v3.z; acc[15] += v3.w;
        }
      }
    }
    float* out = p.partial + static_cast<int64_t>(chunk) * T * p.N + n;
#pragma unroll
    for (int t = 0; t < 16; ++t)
      if (t < T) out[static_cast<int64_t>(t) * p.N] = acc[t];
  }
}

size_t lut_smem_bytes(int J, int M, int Tp, int T) {
  return static_cast<size_t>(J) * M * 256 * Tp * 4 + static_cast<size_t>(T) * J * 8 * 4;
}

cudaError_t launch_lut(const LutParams& p, cudaStream_t st) {
  static std::atomic<int> configured[64] = {};
  const size_t bytes = lut_smem_bytes(p.J, p.M, p.Tp, p.T);
  const cudaError_t se = ensure_dynamic_smem(lut_kernel, bytes, configured);
  if (se != cudaSuccess) return se;
  const int n_slices = (p.N + p.rows_per_cta - 1) / p.rows_per_cta;
  dim3 grid(p.chunks, n_slices);
  return launch_pdl(lut_kernel, grid, dim3(256), bytes, st, p);
}

}  // namespace aq
