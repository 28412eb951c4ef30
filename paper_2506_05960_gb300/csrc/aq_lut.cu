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

// Up to four tokens (TP = 1, 2 or 4 floats per table entry; T <= TP): the same order with
// chunks of whole packed K blocks and at most 64 KB of tables, and one thread per output row:
// per K block it reads the row's 8 * M codes as M contiguous 8-byte pieces (consecutive rows
// consecutive, so a warp's loads are coalesced) and adds, per code, the entry's TP floats with
// one vector load, in the fixed order (K block, group, codebook).  MM: M when 1, 2 or 4 (index
// arithmetic known at compile time; then a chunk is 8 / (MM * TP) K blocks, at least one, and
// the row's code pieces are loaded together, the next row's while this row's entries are
// summed), or 0: any M, one token.
template <int MM, int TP>
__global__ void __launch_bounds__(256) lutv_kernel(const LutParams p) {
  extern __shared__ float4 lut_smem4[];
  float* L = reinterpret_cast<float*>(lut_smem4);              // [J][M][256][TP]
  const int J = p.J, M = MM > 0 ? MM : p.M, T = p.T;
  float* xs = L + static_cast<size_t>(J) * M * 256 * TP;       // [TP][J * 8]
  grid_dependency_wait();
  allow_dependents();
  const int chunk = blockIdx.x;
  const int g0 = chunk * J;
  const int nj = min(J, p.G - g0);
  const int width = J * 8;
  for (int i = threadIdx.x; i < TP * width; i += blockDim.x) {
    const int t = i / width;
    const int e = i - t * width;
    xs[i] = (t < T && e < nj * 8)
                ? static_cast<float>(p.xq[static_cast<int64_t>(t) * p.K + g0 * 8 + e])
                : 0.0f;
  }
  __syncthreads();
  // build: L[j][m][c][t] = sum_e x[t][g0 + j][e] * C^(m)[c][e], ascending e (zero past the last
  // group and past the last token)
  const int entries = J * M * 256;
  for (int ent = threadIdx.x; ent < entries; ent += blockDim.x) {
    const int j = ent / (M * 256);
    const int r = ent - j * (M * 256);
    const uint4 raw = reinterpret_cast<const uint4*>(p.books)[r];
    const __half2* h2 = reinterpret_cast<const __half2*>(&raw);
    float cw[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __half22float2(h2[i]);
      cw[2 * i] = f.x;
      cw[2 * i + 1] = f.y;
    }
    float o[TP];
#pragma unroll
    for (int t = 0; t < TP; ++t) {
      const float* xr = xs + t * width + j * 8;
      float s = 0.0f;
#pragma unroll
      for (int e = 0; e < 8; ++e) s = fmaf(xr[e], cw[e], s);
      o[t] = s;
    }
    if constexpr (TP == 1) {
      L[ent] = o[0];
    } else if constexpr (TP == 2) {
      reinterpret_cast<float2*>(L)[ent] = make_float2(o[0], o[1]);
    } else {
      reinterpret_cast<float4*>(L)[ent] = make_float4(o[0], o[1], o[2], o[3]);
    }
  }
  __syncthreads();
  const int kb0 = g0 >> 3;
  const int nkb = (nj + 7) >> 3;                  // packed K blocks holding this chunk's groups
  const int n_begin = blockIdx.y * p.rows_per_cta;
  const int n_end = min(p.N, n_begin + p.rows_per_cta);
  if constexpr (MM > 0) {
    constexpr int kBlocks = (MM * TP >= 8) ? 1 : 8 / (MM * TP);
    constexpr int kPieces = kBlocks * MM;         // 8-byte code pieces of a row in a chunk
    auto load = [&](int n, uint2 (&v)[kPieces]) {
#pragma unroll
      for (int b = 0; b < kBlocks; ++b) {
        const uint2* rec = reinterpret_cast<const uint2*>(
            p.packed + (static_cast<int64_t>(kb0 + b) * p.N + n) * 8 * MM);
#pragma unroll
        for (int pc = 0; pc < MM; ++pc)
          v[b * MM + pc] = b < nkb ? __ldcs(rec + pc) : make_uint2(0u, 0u);
      }
    };
    uint2 cur[kPieces], nxt[kPieces];
    int n = n_begin + threadIdx.x;
    if (n < n_end) load(n, cur);
    for (; n < n_end; n += blockDim.x) {
      if (n + static_cast<int>(blockDim.x) < n_end) load(n + blockDim.x, nxt);
      float acc[TP];
#pragma unroll
      for (int t = 0; t < TP; ++t) acc[t] = 0.0f;
#pragma unroll
      for (int b = 0; b < kBlocks; ++b) {
        if (b < nkb) {
          const float* Lb = L + b * 8 * MM * 256 * TP;   // tables of this K block's 8 groups
#pragma unroll
          for (int pc = 0; pc < MM; ++pc) {
            const uint2 v = cur[b * MM + pc];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              // byte pc*8 + k of the record is group (pc*8 + k) / MM, codebook (pc*8 + k) % MM,
              // and its entry is ((pc*8 + k) * 256 + code) of this K block's [8][MM][256]
              const uint32_t code = ((k < 4 ? v.x : v.y) >> (8 * (k & 3))) & 0xFFu;
              const float* e = Lb + ((pc * 8 + k) * 256 + code) * TP;
              if constexpr (TP == 1) {
                acc[0] += e[0];
              } else if constexpr (TP == 2) {
                const float2 w = *reinterpret_cast<const float2*>(e);
                acc[0] += w.x;
                acc[1] += w.y;
              } else {
                const float4 w = *reinterpret_cast<const float4*>(e);
                acc[0] += w.x;
                acc[1] += w.y;
                acc[2] += w.z;
                acc[3] += w.w;
              }
            }
          }
        }
      }
#pragma unroll
      for (int t = 0; t < TP; ++t)
        if (t < T) p.partial[(static_cast<int64_t>(chunk) * T + t) * p.N + n] = acc[t];
#pragma unroll
      for (int i = 0; i < kPieces; ++i) cur[i] = nxt[i];
    }
  } else {
    static_assert(MM > 0 || TP == 1, "any M: one token only");
    for (int n = n_begin + threadIdx.x; n < n_end; n += blockDim.x) {
      float acc = 0.0f;
      for (int b = 0; b < nkb; ++b) {
        const uint2* rec = reinterpret_cast<const uint2*>(
            p.packed + (static_cast<int64_t>(kb0 + b) * p.N + n) * 8 * M);
        const float* Lb = L + b * 8 * M * 256;      // tables of this K block's 8 groups
        for (int pc = 0; pc < M; ++pc) {
          const uint2 v = __ldcs(rec + pc);         // streamed once: no reuse in L1
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t code = ((k < 4 ? v.x : v.y) >> (8 * (k & 3))) & 0xFFu;
            acc += Lb[(pc * 8 + k) * 256 + code];
          }
        }
      }
      p.partial[static_cast<int64_t>(chunk) * p.N + n] = acc;
    }
  }
}

size_t lut_smem_bytes(int J, int M, int Tp, int T) {
  return static_cast<size_t>(J) * M * 256 * Tp * 4 + static_cast<size_t>(T) * J * 8 * 4;
}

cudaError_t launch_lut(const LutParams& p, cudaStream_t st) {
  if (p.vec) {
    // lutv_kernel: whole K blocks per chunk, TP = p.Tp floats per entry
    static std::atomic<int> c11[64] = {}, c21[64] = {}, c41[64] = {}, c01[64] = {}, c12[64] = {},
                            c22[64] = {}, c42[64] = {}, c14[64] = {}, c24[64] = {}, c44[64] = {};
    const size_t bytes = static_cast<size_t>(p.J) * p.M * 256 * p.Tp * 4 +
                         static_cast<size_t>(p.Tp) * p.J * 8 * 4;
    const int n_slices = (p.N + p.rows_per_cta - 1) / p.rows_per_cta;
    const dim3 grid(p.chunks, n_slices);
    auto go = [&](auto kernel, std::atomic<int> (&conf)[64]) -> cudaError_t {
      const cudaError_t se = ensure_dynamic_smem(kernel, bytes, conf);
      if (se != cudaSuccess) return se;
      return launch_pdl(kernel, grid, dim3(256), bytes, st, p);
    };
    const int mm = (p.M == 1 || p.M == 2 || p.M == 4) ? p.M : 0;
    switch (p.Tp * 16 + mm) {
      case 16 + 1: return go(lutv_kernel<1, 1>, c11);
      case 16 + 2: return go(lutv_kernel<2, 1>, c21);
      case 16 + 4: return go(lutv_kernel<4, 1>, c41);
      case 16 + 0: return go(lutv_kernel<0, 1>, c01);
      case 32 + 1: return go(lutv_kernel<1, 2>, c12);
      case 32 + 2: return go(lutv_kernel<2, 2>, c22);
      case 32 + 4: return go(lutv_kernel<4, 2>, c42);
      case 64 + 1: return go(lutv_kernel<1, 4>, c14);
      case 64 + 2: return go(lutv_kernel<2, 4>, c24);
      case 64 + 4: return go(lutv_kernel<4, 4>, c44);
      default: return cudaErrorInvalidConfiguration;
    }
  }
  static std::atomic<int> configured[64] = {};
  const size_t bytes = lut_smem_bytes(p.J, p.M, p.Tp, p.T);
  const cudaError_t se = ensure_dynamic_smem(lut_kernel, bytes, configured);
  if (se != cudaSuccess) return se;
  const int n_slices = (p.N + p.rows_per_cta - 1) / p.rows_per_cta;
  dim3 grid(p.chunks, n_slices);
  return launch_pdl(lut_kernel, grid, dim3(256), bytes, st, p);
}

}  // namespace aq
