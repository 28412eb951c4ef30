// aq_codec.cu -- memory-bound kernels of the AQ x A8 layer:
//   * 8-bit activation quantizer (Sec. 4.2.3, symmetric form of Eq. 3)
//   * code packing into the 64-wide-K-block layout
//   * AQ decode (Sec. 2.4 Eq. 4): W-hat = sum of the selected codewords, fp32
//     sum in ascending codebook order, one round to fp16.
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"
#include "aq_quant.cuh"

namespace aq {

// ============================================================== quantizer (rule in aq_quant.cuh)
// Each thread: 16 elements (32 B in; 16 B of int8 codes out, or 32 B with each code stored
// as the fp16 value of that integer, kF16Out) per grid-stride step over `nblocks` blocks
// (block index `bid`); the first block also takes the scalar tail (numel % 16 elements).
template <bool kF16Out>
__device__ __forceinline__ void quant_range(const __half* __restrict__ x, void* __restrict__ out,
                                            int64_t nvec, int64_t numel, float s, int bid,
                                            int nblocks) {
  const float rs = __frcp_rn(s);
  const int64_t stride = static_cast<int64_t>(nblocks) * blockDim.x;
  for (int64_t v = static_cast<int64_t>(bid) * blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const uint4* src = reinterpret_cast<const uint4*>(x) + 2 * v;
    uint4 a = __ldcs(src);
    uint4 b = __ldcs(src + 1);
    __half2 h[8];
    *reinterpret_cast<uint4*>(&h[0]) = a;
    *reinterpret_cast<uint4*>(&h[4]) = b;
    // all 16 values on the fast path (FMA/ALU pipes, straight-line); a value near a tie
    // is redone alone with the exact rule
    uint32_t qb[16];
    bool fast = true;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float2 xf = __half22float2(h[i]);
      fast &= quant_fast_bits(xf.x, rs, qb[2 * i]);
      fast &= quant_fast_bits(xf.y, rs, qb[2 * i + 1]);
    }
    if (!fast) quant_fix16(h, qb, s, rs);
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
      w[i] = pack_low_bytes(qb[4 * i], qb[4 * i + 1], qb[4 * i + 2], qb[4 * i + 3]);
    if constexpr (kF16Out) {
      // int8 -> fp16 is exact (|code| <= 127)
      uint32_t f[8];
#pragma unroll
      for (int i = 0; i < 4; ++i) i8x4_to_f16x4(w[i], f[2 * i], f[2 * i + 1]);
      uint4* dst = reinterpret_cast<uint4*>(out) + 2 * v;
      __stcs(dst, make_uint4(f[0], f[1], f[2], f[3]));
      __stcs(dst + 1, make_uint4(f[4], f[5], f[6], f[7]));
    } else {
      __stcs(reinterpret_cast<uint4*>(out) + v, make_uint4(w[0], w[1], w[2], w[3]));
    }
  }
  if (bid == 0) {
    for (int64_t i = nvec * 16 + threadIdx.x; i < numel; i += blockDim.x) {
      const int8_t c = quant_one(x[i], s, rs);
      if constexpr (kF16Out)
        static_cast<__half*>(out)[i] = __short2half_rn(static_cast<short>(c));
      else
        static_cast<int8_t*>(out)[i] = c;
    }
  }
}

template <bool kF16Out>
__global__ void __launch_bounds__(256) quant_act_kernel(const __half* __restrict__ x,
                                                        void* __restrict__ out,
                                                        int64_t nvec, int64_t numel, float s) {
  grid_dependency_wait();
  allow_dependents();
  quant_range<kF16Out>(x, out, nvec, numel, s, blockIdx.x, gridDim.x);
}

static cudaError_t launch_quant(const void* x, void* out, int64_t numel, float s, bool f16_out,
                                cudaStream_t st) {
  const int64_t nvec = numel / 16;
  int64_t blocks = (nvec + 255) / 256;
  const int64_t cap = 152 * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  auto kernel = f16_out ? quant_act_kernel<true> : quant_act_kernel<false>;
  return launch_pdl(kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st,
                    static_cast<const __half*>(x), out, nvec, numel, s);
}

cudaError_t launch_quant_act(const void* x, int8_t* xq, int64_t numel, float s,
                             cudaStream_t st) {
  return launch_quant(x, xq, numel, s, false, st);
}

cudaError_t launch_quant_act_f16(const void* x, __half* xh, int64_t numel, float s,
                                 cudaStream_t st) {
  return launch_quant(x, xh, numel, s, true, st);
}

// ============================================================== packing
// canonical [N][G][M] (elem bytes eb) -> packed [KB][N][8][M]; one thread per (kb, n).
__global__ void pack_kernel(const uint8_t* __restrict__ canon, uint8_t* __restrict__ packed,
                            int N, int G, int M, int eb, int KB) {
  grid_dependency_wait();
  allow_dependents();
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= static_cast<int64_t>(KB) * N) return;
  const int kb = static_cast<int>(idx / N);
  const int n = static_cast<int>(idx % N);
  const int row_bytes = 8 * M * eb;                    // packed bytes of one (kb, n)
  const int g0 = kb * 8;
  const int ng = min(8, G - g0);
  const uint8_t* src = canon + (static_cast<int64_t>(n) * G + g0) * M * eb;
  uint8_t* dst = packed + idx * row_bytes;
  const int valid = ng * M * eb;
  for (int i = 0; i < row_bytes; ++i) dst[i] = (i < valid) ? src[i] : 0;
}

cudaError_t launch_pack(const void* canon, void* packed, int N, int K, int M, int B,
                        cudaStream_t st) {
  const int G = K / 8;
  const int KB = (K + 63) / 64;
  const int64_t total = static_cast<int64_t>(KB) * N;
  const int threads = 256;
  const int64_t blocks = (total + threads - 1) / threads;
  return launch_pdl(pack_kernel, dim3(static_cast<unsigned>(blocks)), dim3(threads), 0, st,
                    static_cast<const uint8_t*>(canon), static_cast<uint8_t*>(packed), N, G, M,
                    B / 8, KB);
}

// ============================================================== decode
// Sum of M codewords of one group in fp32, ascending m, one RNE to fp16.
// cw(m) returns the 16-byte codeword of codebook m.
struct F8 {
  float v[8];
};

__device__ __forceinline__ void widen_add(F8& acc, const uint4& cw, bool first) {
  const __half2* h = reinterpret_cast<const __half2*>(&cw);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __half22float2(h[i]);
    if (first) {
      acc.v[2 * i] = f.x;
      acc.v[2 * i + 1] = f.y;
    } else {
      acc.v[2 * i] = __fadd_rn(acc.v[2 * i], f.x);
      acc.v[2 * i + 1] = __fadd_rn(acc.v[2 * i + 1], f.y);
    }
  }
}

__device__ __forceinline__ uint4 narrow(const F8& acc) {
  uint4 r;
  uint32_t* p = reinterpret_cast<uint32_t*>(&r);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    __half2 h = __floats2half2_rn(acc.v[2 * i], acc.v[2 * i + 1]);
    p[i] = *reinterpret_cast<uint32_t*>(&h);
  }
  return r;
}

// 8-bit codes: all M codebooks (M x 256 x 16 B <= 32 KB) staged in shared memory by the
// caller.  One thread per group: packed index idx = (kb*N + n)*8 + j is also the
// thread's linear index, so code loads are contiguous across the warp and each group of
// 8 threads writes 128 contiguous bytes of W.
__device__ __forceinline__ void decode_b8_range(const uint8_t* __restrict__ packed,
                                                const uint4* sbook, __half* __restrict__ W,
                                                int N, int K, int M, int KB, int bid,
                                                int nblocks) {
  const int G = K / 8;
  const int64_t total = static_cast<int64_t>(KB) * N * 8;
  for (int64_t idx = static_cast<int64_t>(bid) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(nblocks) * blockDim.x) {
    const int j = static_cast<int>(idx & 7);
    const int64_t rem = idx >> 3;
    const int kb = static_cast<int>(rem / N);
    const int n = static_cast<int>(rem - static_cast<int64_t>(kb) * N);
    const int grp = kb * 8 + j;
    if (grp >= G) continue;
    const uint8_t* c = packed + idx * M;
    F8 acc;
    for (int m = 0; m < M; ++m) widen_add(acc, sbook[m * 256 + c[m]], m == 0);
    *reinterpret_cast<uint4*>(W + static_cast<int64_t>(n) * K + grp * 8) = narrow(acc);
  }
}

// 16-bit codes: codebooks (M x 65536 x 16 B) stay in global memory / L2.
__device__ __forceinline__ void decode_b16_range(const uint16_t* __restrict__ packed,
                                                 const uint4* __restrict__ books,
                                                 __half* __restrict__ W, int N, int K, int M,
                                                 int KB, int bid, int nblocks) {
  const int G = K / 8;
  const int64_t total = static_cast<int64_t>(KB) * N * 8;
  for (int64_t idx = static_cast<int64_t>(bid) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(nblocks) * blockDim.x) {
    const int j = static_cast<int>(idx & 7);
    const int64_t rem = idx >> 3;
    const int kb = static_cast<int>(rem / N);
    const int n = static_cast<int>(rem - static_cast<int64_t>(kb) * N);
    const int grp = kb * 8 + j;
    if (grp >= G) continue;
    const uint16_t* c = packed + idx * M;
    F8 acc;
    for (int m = 0; m < M; ++m)
      widen_add(acc, __ldg(books + (static_cast<int64_t>(m) << 16) + c[m]), m == 0);
    *reinterpret_cast<uint4*>(W + static_cast<int64_t>(n) * K + grp * 8) = narrow(acc);
  }
}

__device__ __forceinline__ void stage_books8(const uint4* __restrict__ books, uint4* sbook, int M) {
  for (int i = threadIdx.x; i < M * 256; i += blockDim.x) sbook[i] = books[i];
  __syncthreads();
}

__global__ void __launch_bounds__(512) decode_b8_kernel(const uint8_t* __restrict__ packed,
                                                        const uint4* __restrict__ books,
                                                        __half* __restrict__ W, int N, int K,
                                                        int M, int KB) {
  extern __shared__ uint4 sbook[];                       // [M][256]
  if (threadIdx.x == 0) {
    // the codes and books do not come from the previous kernel: this block's first codes
    // start moving into L2 while it still runs (a hint, no effect on memory values)
    const int64_t total = static_cast<int64_t>(KB) * N * 8 * M;
    const int64_t first = static_cast<int64_t>(blockIdx.x) * blockDim.x * M;
    const int64_t left = total - first;
    const int64_t span = left < static_cast<int64_t>(blockDim.x) * M ? left : blockDim.x * M;
    const uint32_t bytes = static_cast<uint32_t>(span > 0 ? span : 0) & ~15u;
    if (bytes > 0) bulk_prefetch_l2(packed + first, bytes);
    if (blockIdx.x == 0) bulk_prefetch_l2(books, static_cast<uint32_t>(M * 256 * 16));
  }
  grid_dependency_wait();
  allow_dependents();
  stage_books8(books, sbook, M);
  decode_b8_range(packed, sbook, W, N, K, M, KB, blockIdx.x, gridDim.x);
}

__global__ void __launch_bounds__(512) decode_b16_kernel(const uint16_t* __restrict__ packed,
                                                         const uint4* __restrict__ books,
                                                         __half* __restrict__ W, int N, int K,
                                                         int M, int KB) {
  grid_dependency_wait();
  allow_dependents();
  decode_b16_range(packed, books, W, N, K, M, KB, blockIdx.x, gridDim.x);
}

cudaError_t launch_decode(const void* packed, const void* books, void* W, int N, int K, int M,
                          int B, cudaStream_t st) {
  const int KB = (K + 63) / 64;
  const int64_t total = static_cast<int64_t>(KB) * N * 8;
  const int threads = 512;
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > 152 * 4) blocks = 152 * 4;
  if (blocks < 1) blocks = 1;
  if (B == 8)
    return launch_pdl(decode_b8_kernel, dim3(static_cast<unsigned>(blocks)), dim3(threads),
                      static_cast<size_t>(M) * 256 * 16, st, static_cast<const uint8_t*>(packed),
                      static_cast<const uint4*>(books), static_cast<__half*>(W), N, K, M, KB);
  return launch_pdl(decode_b16_kernel, dim3(static_cast<unsigned>(blocks)), dim3(threads), 0, st,
                    static_cast<const uint16_t*>(packed), static_cast<const uint4*>(books),
                    static_cast<__half*>(W), N, K, M, KB);
}

// ============================================================== transposed, scaled decode
// For the input gradient of the layer (Sec. 3.2.1's continuous step back-propagates through
// it): dX[t][k] = alpha * sum_n dY[t][n] * scale[n] * W[n][k] = alpha * (dY Wt^T)[t][k] with
// Wt[k][n] = fp16(scale[n] * W[n][k]): W[n][k] decoded by the rule of Eq. 4 (fp32 sum in
// ascending m, one round to fp16), times the fp16 scale in fp32, one more round to fp16.
// CTA = 64 output rows n x one 64-wide K block, thread = one (n, group j): it decodes its
// group and writes the 8 scaled values down a column of a transposed shared-memory tile
// [64 k][64 n] (rows padded to 66 halves); the tile's rows (64 n values, 128 B each) are
// then written to Wt.  Block (0, 0) also writes `ones` (K fp16 ones, the unit per-column
// scale of the gradient GEMM's epilogue).
constexpr int kTRows = 64;                     // output rows n per CTA
constexpr int kTPad = 66;                      // tile row stride in halves

template <int EB>
__global__ void __launch_bounds__(512) decode_t_kernel(const void* __restrict__ packed,
                                                       const uint4* __restrict__ books,
                                                       const __half* __restrict__ scale,
                                                       __half* __restrict__ Wt, __half* ones,
                                                       int N, int K, int M) {
  __shared__ __half tile[64 * kTPad];
  grid_dependency_wait();
  allow_dependents();
  const int kb = blockIdx.y;
  const int n0 = blockIdx.x * kTRows;
  const int nl = threadIdx.x >> 3, j = threadIdx.x & 7;
  const int n = n0 + nl;
  const int G = K / 8;
  const int grp = kb * 8 + j;
  if (blockIdx.x == 0 && blockIdx.y == 0)
    for (int i = threadIdx.x; i < K; i += blockDim.x) ones[i] = __float2half_rn(1.0f);
  float v[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  if (n < N && grp < G) {
    const int64_t idx = (static_cast<int64_t>(kb) * N + n) * 8 + j;
    F8 acc;
    for (int m = 0; m < M; ++m) {
      const uint32_t c = EB == 1 ? static_cast<const uint8_t*>(packed)[idx * M + m]
                                 : static_cast<const uint16_t*>(packed)[idx * M + m];
      widen_add(acc, __ldg(books + (static_cast<int64_t>(m) << (8 * EB)) + c), m == 0);
    }
    const uint4 w = narrow(acc);               // the decoded weight, fp16 (Eq. 4 rule)
    const float sc = __half2float(scale[n]);
    const __half2* h = reinterpret_cast<const __half2*>(&w);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __half22float2(h[i]);
      v[2 * i] = __fmul_rn(f.x, sc);
      v[2 * i + 1] = __fmul_rn(f.y, sc);
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) tile[(j * 8 + e) * kTPad + nl] = __float2half_rn(v[e]);
  __syncthreads();
  // row r of the tile = k = kb*64 + r, columns n0 .. n0+63: 8 chunks of 8 halves
  const int r = threadIdx.x >> 3, ch = threadIdx.x & 7;
  const int k = kb * 64 + r;
  const int nc = n0 + ch * 8;
  if (k < K && nc < N) {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(tile + r * kTPad + ch * 8);
    const uint4 out = make_uint4(src[0], src[1], src[2], src[3]);
    *reinterpret_cast<uint4*>(Wt + static_cast<int64_t>(k) * N + nc) = out;   // N % 8 == 0
  }
}

cudaError_t launch_decode_t(const void* packed, const void* books, const __half* scale,
                            __half* Wt, __half* ones, int N, int K, int M, int B,
                            cudaStream_t st) {
  const dim3 grid(static_cast<unsigned>((N + kTRows - 1) / kTRows),
                  static_cast<unsigned>((K + 63) / 64));
  if (B == 8)
    return launch_pdl(decode_t_kernel<1>, grid, dim3(512), 0, st, packed,
                      static_cast<const uint4*>(books), scale, Wt, ones, N, K, M);
  return launch_pdl(decode_t_kernel<2>, grid, dim3(512), 0, st, packed,
                    static_cast<const uint4*>(books), scale, Wt, ones, N, K, M);
}

// ============================================================== kernel-aware decode (g = 9)
// Sec. 3.1.2 / App. A.1 Eq. A4: one group = the 3x3 taps of one (output channel n,
// input channel c) filter; codes [N][Cin][M], codebooks [M][2^B][9] fp16.  The
// decoded filter is written in the K order of the implicit-GEMM convolution,
// W[n][t*Cin + c] for tap t = i*3 + j, so the tensor-core path is unchanged.  Same
// rule as the 8-wide decode: fp32 sum in ascending m, one RNE to fp16.  One thread
// per (n, c): consecutive threads take consecutive c, so each tap's stores are
// contiguous across the warp.  8-bit books are staged in shared memory.
template <int EB>
__global__ void __launch_bounds__(256) decode_kaq_kernel(const uint8_t* __restrict__ codes,
                                                         const __half* __restrict__ books,
                                                         __half* __restrict__ W, int N, int Cin,
                                                         int M) {
  extern __shared__ __half sbook9[];                     // [M][256][9] for 8-bit codes
  grid_dependency_wait();
  allow_dependents();
  if constexpr (EB == 1) {
    for (int i = threadIdx.x; i < M * 256 * 9; i += blockDim.x) sbook9[i] = books[i];
    __syncthreads();
  }
  const int K = 9 * Cin;
  const int64_t total = static_cast<int64_t>(N) * Cin;
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int n = static_cast<int>(idx / Cin);
    const int c = static_cast<int>(idx - static_cast<int64_t>(n) * Cin);
    float acc[9];
    for (int m = 0; m < M; ++m) {
      const __half* cw;
      if constexpr (EB == 1) {
        cw = sbook9 + (m * 256 + codes[idx * M + m]) * 9;
      } else {
        const uint16_t b = reinterpret_cast<const uint16_t*>(codes)[idx * M + m];
        cw = books + ((static_cast<int64_t>(m) << 16) + b) * 9;
      }
#pragma unroll
      for (int t = 0; t < 9; ++t) {
        const float v = __half2float(EB == 1 ? cw[t] : __ldg(cw + t));
        acc[t] = m == 0 ? v : __fadd_rn(acc[t], v);
      }
    }
    __half* out = W + static_cast<int64_t>(n) * K + c;
#pragma unroll
    for (int t = 0; t < 9; ++t) out[static_cast<int64_t>(t) * Cin] = __float2half_rn(acc[t]);
  }
}

cudaError_t launch_decode_kaq(const void* codes, const void* books, void* W, int N, int Cin, int M,
                              int B, cudaStream_t st) {
  const int64_t total = static_cast<int64_t>(N) * Cin;
  int64_t blocks = (total + 255) / 256;
  const int64_t cap = B == 8 ? 152 * 2 : 152 * 8;       // 8-bit: every block stages the books
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  const uint8_t* c = static_cast<const uint8_t*>(codes);
  const __half* b = static_cast<const __half*>(books);
  __half* w = static_cast<__half*>(W);
  if (B == 8)
    return launch_pdl(decode_kaq_kernel<1>, dim3(static_cast<unsigned>(blocks)), dim3(256),
                      static_cast<size_t>(M) * 256 * 9 * 2, st, c, b, w, N, Cin, M);
  return launch_pdl(decode_kaq_kernel<2>, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, c,
                    b, w, N, Cin, M);
}

// ============================================================== codebook gradient
// Backward of Eq. 4 for the continuous (codebook) step of Stage-2 fine-tuning
// (Sec. 3.2.1, PV-Tuning): the decoded group is sum_m C^(m)[b_m], so
//   dL/dC^(m)[c][e] = sum over groups (n, i) with b[n][i][m] = c of
//                     s_x * scale[n] * G[n][i*g + e],
// where G[n][k] = sum_t dY[t][n] * xq[t][k] is the gradient with respect to the
// unscaled weight (a plain GEMM the caller runs).  dC is accumulated (+=) in fp32:
// 8-bit codebooks in shared memory per CTA, flushed with global atomics; 16-bit
// codebooks with global atomics directly.  One thread per group (its G row piece and
// its M codes are loaded before the first add); g = 8 reads the packed layout, g = 9
// (one group per 3x3 filter) the canonical [N][Cin][M] codes with G in the
// convolution's OHWI order.
template <int EB, bool kKaq>
__global__ void __launch_bounds__(256, 2) codebook_grad_kernel(
    const uint8_t* __restrict__ codes, const float* __restrict__ G,
    const __half* __restrict__ scale, float s_x, float* __restrict__ dC, int N, int K, int M,
    int KB) {
  constexpr int g = kKaq ? 9 : 8;
  constexpr int kMaxM = EB == 1 ? 8 : 2;
  // 8-bit codes: the CTA's table in shared memory, element-major [g][M*256] so that
  // the adds of a warp (random codewords, same element) spread over all banks
  extern __shared__ float sdc[];
  grid_dependency_wait();
  allow_dependents();
  if constexpr (EB == 1) {
    for (int i = threadIdx.x; i < M * 256 * g; i += blockDim.x) sdc[i] = 0.0f;
    __syncthreads();
  }
  const int Cin = K / 9;
  const int64_t total = kKaq ? static_cast<int64_t>(N) * Cin : static_cast<int64_t>(KB) * N * 8;
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    int n, col0, colstep;
    if constexpr (kKaq) {
      n = static_cast<int>(idx / Cin);
      const int c = static_cast<int>(idx - static_cast<int64_t>(n) * Cin);
      col0 = c;
      colstep = Cin;                                    // tap t at t*Cin + c
    } else {
      const int j = static_cast<int>(idx & 7);
      const int64_t r = idx >> 3;
      const int kb = static_cast<int>(r / N);
      n = static_cast<int>(r - static_cast<int64_t>(kb) * N);
      col0 = (kb * 8 + j) * 8;
      colstep = 1;
      if (col0 >= K) continue;                          // zero-padded K tail
    }
    const float f = s_x * (scale ? __half2float(scale[n]) : 1.0f);
    const float* grow = G + static_cast<int64_t>(n) * K + col0;
    float v[g];
    if constexpr (kKaq) {
#pragma unroll
      for (int e = 0; e < g; ++e) v[e] = f * __ldg(grow + static_cast<int64_t>(e) * colstep);
    } else {
      // 8 consecutive floats of the row (32-byte aligned: K % 8 == 0, G 16-byte aligned)
      const float4 a = __ldg(reinterpret_cast<const float4*>(grow));
      const float4 b = __ldg(reinterpret_cast<const float4*>(grow) + 1);
      v[0] = f * a.x; v[1] = f * a.y; v[2] = f * a.z; v[3] = f * a.w;
      v[4] = f * b.x; v[5] = f * b.y; v[6] = f * b.z; v[7] = f * b.w;
    }
    int cw[kMaxM];
#pragma unroll
    for (int m = 0; m < kMaxM; ++m)
      if (m < M)
        cw[m] = EB == 1 ? codes[idx * M + m]
                        : reinterpret_cast<const uint16_t*>(codes)[idx * M + m];
#pragma unroll
    for (int m = 0; m < kMaxM; ++m) {
      if (m >= M) break;
      if constexpr (EB == 1) {
        float* dst = sdc + m * 256 + cw[m];
#pragma unroll
        for (int e = 0; e < g; ++e) atomicAdd(dst + e * (M * 256), v[e]);
      } else {
        float* dst = dC + ((static_cast<int64_t>(m) << 16) + cw[m]) * g;
#pragma unroll
        for (int e = 0; e < g; ++e) atomicAdd(dst + e, v[e]);
      }
    }
  }
  if constexpr (EB == 1) {
    // flush: dC[m][c][e] += table[e][m*256 + c], 4 consecutive entries per vector atomic
    // (M*256*g is a multiple of 4; dC is 16-byte aligned)
    __syncthreads();
    for (int i = threadIdx.x; i < M * 256 * g / 4; i += blockDim.x) {
      float w[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int lin = 4 * i + u;                      // = (m*256 + c)*g + e
        const int mc = lin / g;
        w[u] = sdc[(lin - mc * g) * (M * 256) + mc];
      }
      if (w[0] != 0.0f || w[1] != 0.0f || w[2] != 0.0f || w[3] != 0.0f)
        asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(dC + 4 * i),
                     "f"(w[0]), "f"(w[1]), "f"(w[2]), "f"(w[3])
                     : "memory");
    }
  }
}

cudaError_t launch_codebook_grad(const void* codes, const float* G, const __half* scale,
                                 float s_x, float* dC, int N, int K, int g, int M, int B,
                                 cudaStream_t st) {
  const bool kaq = g == 9;
  const int KB = (K + 63) / 64;
  const int64_t total = kaq ? static_cast<int64_t>(N) * (K / 9) : static_cast<int64_t>(KB) * N * 8;
  // 8-bit: two blocks per SM, each flushes its table once (more threads per SM only
  // add shared-memory atomic contention; a flush summed first over a cluster's tables
  // through distributed shared memory measured slower)
  const int threads = 256;
  const int64_t cap = B == 8 ? 152 * 2 : 152 * 8;
  int64_t blocks = (total + threads - 1) / threads;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  const dim3 grid(static_cast<unsigned>(blocks)), block(static_cast<unsigned>(threads));
  const uint8_t* c = static_cast<const uint8_t*>(codes);
  const size_t smem = B == 8 ? static_cast<size_t>(M) * 256 * g * 4 : 0;
  if (B == 8) {
    auto kernel = kaq ? codebook_grad_kernel<1, true> : codebook_grad_kernel<1, false>;
    if (smem > 48 * 1024)
      cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem));
    return launch_pdl(kernel, grid, block, smem, st, c, G, scale, s_x, dC, N, K, M, KB);
  }
  if (kaq)
    return launch_pdl(codebook_grad_kernel<2, true>, grid, block, 0, st, c, G, scale, s_x, dC, N,
                      K, M, KB);
  return launch_pdl(codebook_grad_kernel<2, false>, grid, block, 0, st, c, G, scale, s_x, dC, N,
                    K, M, KB);
}

// ============================================================== code search step
// Stage-1 calibration (Sec. 3.1; the code optimisation of AQLM, beam width 1): for
// every group and each codebook m in [m_first, m_first + m_count) in turn, set
// b[m] to the codeword minimising the group's error with the other codewords fixed:
//   r = w - sum_{m' != m} C^(m')[b[m']] (ascending m'),  d = C^(m)[c] - r,
//   score(c) = d^T H d  (H = the group's 8x8 block of A A^T, or I when H is NULL),
// in fp32 with every product and sum rounded separately in ascending element order
// (no fused multiply-add), ties to the lowest c -- the same decision as the
// reference step.  8-bit codes (256 candidates, codebooks staged in shared memory
// as fp16); one thread per group, consecutive threads on consecutive rows of the
// same group column so that a warp shares H's block.
template <bool kWeighted>
__global__ void __launch_bounds__(256) code_update_kernel(const float* __restrict__ W,
                                                          const __half* __restrict__ books,
                                                          uint8_t* __restrict__ codes,
                                                          const float* __restrict__ H,
                                                          int m_first, int m_count, int N, int K,
                                                          int M) {
  extern __shared__ __half sb[];                          // [M][256][8]
  grid_dependency_wait();
  allow_dependents();
  for (int i = threadIdx.x; i < M * 256 * 8; i += blockDim.x) sb[i] = books[i];
  __syncthreads();
  const int Gr = K / 8;
  const int64_t total = static_cast<int64_t>(N) * Gr;
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(idx / N);
    const int n = static_cast<int>(idx - static_cast<int64_t>(i) * N);
    uint8_t* bc = codes + (static_cast<int64_t>(n) * Gr + i) * M;
    float w[8];
    const float4 w0 = __ldg(reinterpret_cast<const float4*>(W + static_cast<int64_t>(n) * K + i * 8));
    const float4 w1 = __ldg(reinterpret_cast<const float4*>(W + static_cast<int64_t>(n) * K + i * 8) + 1);
    w[0] = w0.x; w[1] = w0.y; w[2] = w0.z; w[3] = w0.w;
    w[4] = w1.x; w[5] = w1.y; w[6] = w1.z; w[7] = w1.w;
    float h[64];
    if constexpr (kWeighted) {
#pragma unroll
      for (int e = 0; e < 64; ++e) h[e] = __ldg(H + i * 64 + e);
    }
    for (int m = m_first; m < m_first + m_count; ++m) {
      float r[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) r[e] = w[e];
      for (int m2 = 0; m2 < M; ++m2) {
        if (m2 == m) continue;
        const __half* cw = sb + (m2 * 256 + bc[m2]) * 8;
#pragma unroll
        for (int e = 0; e < 8; ++e) r[e] = __fsub_rn(r[e], __half2float(cw[e]));
      }
      float best = 0.0f;
      int best_c = 0;
      for (int c = 0; c < 256; ++c) {
        const __half* cw = sb + (m * 256 + c) * 8;
        float d[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) d[e] = __fsub_rn(__half2float(cw[e]), r[e]);
        float sc = 0.0f;
        if constexpr (kWeighted) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            float t = 0.0f;
#pragma unroll
            for (int e2 = 0; e2 < 8; ++e2) t = __fadd_rn(t, __fmul_rn(h[e * 8 + e2], d[e2]));
            sc = __fadd_rn(sc, __fmul_rn(d[e], t));
          }
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) sc = __fadd_rn(sc, __fmul_rn(d[e], d[e]));
        }
        if (c == 0 || sc < best) {
          best = sc;
          best_c = c;
        }
      }
      bc[m] = static_cast<uint8_t>(best_c);
    }
  }
}

cudaError_t launch_code_update(const float* W, const void* books, void* codes, const float* H,
                               int m_first, int m_count, int N, int K, int M, cudaStream_t st) {
  const int64_t total = static_cast<int64_t>(N) * (K / 8);
  int64_t blocks = (total + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  const size_t smem = static_cast<size_t>(M) * 256 * 8 * 2;
  const __half* b = static_cast<const __half*>(books);
  uint8_t* c = static_cast<uint8_t*>(codes);
  if (H)
    return launch_pdl(code_update_kernel<true>, dim3(static_cast<unsigned>(blocks)), dim3(256), smem,
                      st, W, b, c, H, m_first, m_count, N, K, M);
  return launch_pdl(code_update_kernel<false>, dim3(static_cast<unsigned>(blocks)), dim3(256), smem,
                    st, W, b, c, H, m_first, m_count, N, K, M);
}

}  // namespace aq
