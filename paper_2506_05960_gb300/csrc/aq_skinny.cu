// aq_skinny.cu -- the AQ x A8 linear layer for a few tokens (T <= 16), in one pass.
//
// With few tokens the layer is a stream over its packed codes: every weight is decoded
// once (Eq. 4) and used by only T tokens, so the kernel has to read the codes at HBM
// speed and decode them faster than they arrive.  No workspace, no second kernel.
//
// Mapping.  A row block is 8 consecutive output rows.  In a warp, lane 4*r + q owns row
// n0 + r and the groups 2q, 2q+1 of every 64-wide K block, i.e. 16 consecutive k.  The
// packed layout [K/64][N][8][M] keeps the 8 rows' codes of one K block contiguous, so a
// warp reads one 8 * (8 * M)-byte segment per K block (128 B for two 8-bit codes), a
// lane its 2 * M codes in one load.  The CTA's warps take the K blocks round-robin, four
// at a time (their code loads issued before the first lookup).  Each lane decodes its two
// groups -- the fp32 sum of the M codewords in ascending m, one round to fp16; for M <= 2
// the fp16 add gives the same bits (double rounding of a two-term sum through fp32 is
// innocuous) -- and dots the 16 weights with every token's 16 int8 activations in fp32.
// Reduction in a fixed order: the 4 lanes of a row (xor butterflies), then the warps in
// order; the epilogue applies s_x * scale[n] and bias[n] (fp16, fp32, or the next layer's
// int8 activations).  CTAs are persistent over row blocks.
//
// 8-bit codebooks are staged in shared memory in R copies (copy r of entry e in 16-byte
// slot e * R + r, lane l reading copy l % R): the 8 lanes of a quarter warp, whose random
// 16-byte lookups are served together, then always hit 8 different bank groups.  16-bit
// (2^16-entry) codebooks are read from L2 by a second kernel (skinny_gather_kernel, below).
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"
#include "aq_quant.cuh"

namespace aq {

constexpr int kSkinnyRows = 8;    // output rows per row block (lane / 4)
constexpr int kSkinnyWarps = 8;   // warps per CTA; they split the K blocks
constexpr int kSkinnyUnroll = 4;  // K blocks per warp whose code loads are in flight together
constexpr int kSkinnyXsBytes = 32 * 1024;  // activations staged in shared memory up to this size

// 16 int8 (one uint4) -> 16 floats
__device__ __forceinline__ void i8x16_to_f32(uint4 v, float (&x)[16]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int32_t a = static_cast<int32_t>(w[q]);
#pragma unroll
    for (int i = 0; i < 4; ++i) x[4 * q + i] = static_cast<float>((a << (24 - 8 * i)) >> 24);
  }
}

// The 2 * M 8-bit codes of one lane (groups 2q and 2q+1 of a K block, each [M] codes),
// widened to 32 bits: c[i * M + m] = code of codebook m in group 2q + i.
template <int MM>
__device__ __forceinline__ void load_codes(const uint8_t* rec, int q, int M, uint32_t* c) {
  if constexpr (MM == 1) {
    const uint32_t v = *reinterpret_cast<const uint16_t*>(rec + 2 * q);
    c[0] = v & 0xffu;
    c[1] = v >> 8;
  } else if constexpr (MM == 2) {
    const uint32_t v = *reinterpret_cast<const uint32_t*>(rec + 4 * q);
    c[0] = v & 0xffu;
    c[1] = (v >> 8) & 0xffu;
    c[2] = (v >> 16) & 0xffu;
    c[3] = v >> 24;
  } else {
    // any M (3..8): one load per code
    for (int i = 0; i < 2 * M; ++i) c[i] = static_cast<uint32_t>(rec[2 * q * M + i]);
  }
}

// Decoded weights of one group (8 values, the rule of Eq. 4), as fp32, from the shared-
// memory copies of the 8-bit codebooks.
template <int MM>
__device__ __forceinline__ void decode_group(const uint32_t* c, int M, const uint4* sbook, int R,
                                             int copy, float (&w)[8]) {
  auto word = [&](int m) -> uint4 { return sbook[(m * 256 + static_cast<int>(c[m])) * R + copy]; };
  if constexpr (MM == 1 || MM == 2) {
    uint4 v = word(0);
    if constexpr (MM == 2) {
      const uint4 u = word(1);
      __half2* a = reinterpret_cast<__half2*>(&v);
      const __half2* b = reinterpret_cast<const __half2*>(&u);
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = __hadd2(a[i], b[i]);
    }
    const __half2* h = reinterpret_cast<const __half2*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __half22float2(h[i]);
      w[2 * i] = f.x;
      w[2 * i + 1] = f.y;
    }
  } else {
    float s[8];
    for (int m = 0; m < M; ++m) {
      const uint4 v = word(m);
      const __half2* h = reinterpret_cast<const __half2*>(&v);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(h[i]);
        s[2 * i] = m == 0 ? f.x : __fadd_rn(s[2 * i], f.x);
        s[2 * i + 1] = m == 0 ? f.y : __fadd_rn(s[2 * i + 1], f.y);
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e) w[e] = __half2float(__float2half_rn(s[e]));
  }
}

// 8-bit codes.  TT: tokens rounded up to 1, 2, 4, 8 or 16; MM: M when 1 or 2, else 0.
template <int TT, int MM>
__global__ void __launch_bounds__(kSkinnyWarps * 32) skinny_kernel(const SkinnyParams p) {
  extern __shared__ float4 skinny_smem4[];
  const int M = MM > 0 ? MM : p.M;
  const int R = fused_book_copies(M);
  uint4* sbook = reinterpret_cast<uint4*>(skinny_smem4);                   // [M*256][R]
  float* wred = reinterpret_cast<float*>(skinny_smem4) + M * 256 * R * 4;
  // the activations as fp16 (exact for |x| <= 127), [T][K], when p.x_smem: every lane of a
  // row block reads them with broadcast loads instead of converting the same int8 values
  // (one token never stages them: TT == 1 compiles the branch out of the inner loop)
  __half* xs = (TT >= 2 && p.x_smem)
                   ? reinterpret_cast<__half*>(wred + kSkinnyWarps * kSkinnyRows * TT)
                   : nullptr;
  grid_dependency_wait();
  allow_dependents();
  const uint4* gbook = static_cast<const uint4*>(p.books);
  // thread i writes copy (r + i) % R at step r: a quarter warp's stores hit distinct banks
  for (int i = threadIdx.x; i < M * 256; i += blockDim.x) {
    const uint4 v = gbook[i];
    for (int r = 0; r < R; ++r) sbook[i * R + ((r + i) & (R - 1))] = v;
  }
  if (TT >= 2 && xs) {
    // 8 activations (8 bytes, K % 16 == 0 keeps them inside one row) per thread and step
    const int n8 = p.T * p.K / 8;
    for (int i = threadIdx.x; i < n8; i += blockDim.x) {
      const uint2 v = reinterpret_cast<const uint2*>(p.xq)[i];
      uint32_t h0, h1, h2, h3;
      i8x4_to_f16x4(v.x, h0, h1);
      i8x4_to_f16x4(v.y, h2, h3);
      reinterpret_cast<uint4*>(xs)[i] = make_uint4(h0, h1, h2, h3);
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = lane >> 2, q = lane & 3;
  const int copy = lane & (R - 1);
  const int T = p.T, K = p.K, N = p.N;
  const int KB = (K + 63) >> 6;                  // K blocks (the last may be partial)
  const int G = K >> 3;                          // groups; K % 16 == 0, so G is even
  const int CB = 8 * M;                          // code bytes of one row in one K block
  const int n_rb = (N + kSkinnyRows - 1) / kSkinnyRows;
  const uint8_t* codes = static_cast<const uint8_t*>(p.codes);
  const float rs_out = p.out_q8 ? __frcp_rn(p.s_out) : 0.0f;

  for (int rb = blockIdx.x; rb < n_rb; rb += gridDim.x) {
    const int n0 = rb * kSkinnyRows;
    const int n = n0 + r;
    float acc[TT];
#pragma unroll
    for (int t = 0; t < TT; ++t) acc[t] = 0.0f;
    if (n < N) {
      for (int kb0 = warp; kb0 < KB; kb0 += kSkinnyWarps * kSkinnyUnroll) {
        uint32_t c[kSkinnyUnroll][2 * (MM > 0 ? MM : 8)];
        bool ok[kSkinnyUnroll];
#pragma unroll
        for (int u = 0; u < kSkinnyUnroll; ++u) {
          const int kb = kb0 + u * kSkinnyWarps;
          // this lane's two groups exist (G even: both or neither)
          ok[u] = kb < KB && kb * 8 + 2 * q < G;
          if (ok[u])
            load_codes<MM>(codes + (static_cast<int64_t>(kb) * N + n) * CB, q, M, c[u]);
        }
#pragma unroll
        for (int u = 0; u < kSkinnyUnroll; ++u) {
          if (!ok[u]) continue;
          const int kb = kb0 + u * kSkinnyWarps;
          float w[16];
          float (&w0)[8] = *reinterpret_cast<float (*)[8]>(w);
          float (&w1)[8] = *reinterpret_cast<float (*)[8]>(w + 8);
          decode_group<MM>(c[u], M, sbook, R, copy, w0);
          decode_group<MM>(c[u] + M, M, sbook, R, copy, w1);
          const int k0 = kb * 64 + q * 16;
#pragma unroll
          for (int t = 0; t < TT; ++t) {
            if (t < T) {
              float x[16];
              if (TT >= 2 && xs) {
                const uint4* xp = reinterpret_cast<const uint4*>(xs + t * K + k0);
                const uint4 a = xp[0], b = xp[1];
                const __half2* ha = reinterpret_cast<const __half2*>(&a);
                const __half2* hb = reinterpret_cast<const __half2*>(&b);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  const float2 fa = __half22float2(ha[i]);
                  const float2 fb = __half22float2(hb[i]);
                  x[2 * i] = fa.x;
                  x[2 * i + 1] = fa.y;
                  x[8 + 2 * i] = fb.x;
                  x[8 + 2 * i + 1] = fb.y;
                }
              } else {
                i8x16_to_f32(__ldg(reinterpret_cast<const uint4*>(p.xq + static_cast<int64_t>(t) * K + k0)), x);
              }
#pragma unroll
              for (int e = 0; e < 16; ++e) acc[t] = fmaf(w[e], x[e], acc[t]);
            }
          }
        }
      }
    }
    // fixed-order reduction: the 4 lanes of a row, then the warps in order
#pragma unroll
    for (int t = 0; t < TT; ++t) {
      float v = acc[t];
      v += __shfl_xor_sync(0xffffffffu, v, 1);
      v += __shfl_xor_sync(0xffffffffu, v, 2);
      if (q == 0) wred[(warp * kSkinnyRows + r) * TT + t] = v;
    }
    __syncthreads();
    for (int o = threadIdx.x; o < kSkinnyRows * T; o += blockDim.x) {
      const int t = o / kSkinnyRows;
      const int rr = o - t * kSkinnyRows;
      const int nn = n0 + rr;
      if (nn >= N) continue;
      float v = 0.0f;
      for (int wi = 0; wi < kSkinnyWarps; ++wi) v += wred[(wi * kSkinnyRows + rr) * TT + t];
      v = fmaf(v, p.s_x * __half2float(p.scale[nn]), p.bias ? __half2float(p.bias[nn]) : 0.0f);
      const int64_t off = static_cast<int64_t>(t) * N + nn;
      if (p.out_f32)
        static_cast<float*>(p.y)[off] = v;
      else if (p.out_q8 == kOutCodesF16)
        static_cast<__half*>(p.y)[off] =
            __short2half_rn(quant_one(__float2half_rn(v), p.s_out, rs_out));
      else if (p.out_q8)
        static_cast<int8_t*>(p.y)[off] = quant_one(__float2half_rn(v), p.s_out, rs_out);
      else
        static_cast<__half*>(p.y)[off] = __float2half_rn(v);
    }
    __syncthreads();   // wred is rewritten by the next row block
  }
}

// 16-bit codes (2^16-entry codebooks, codewords gathered from L2): four output rows per
// CTA, whose threads stride the K/8 group columns and decode each group for the four rows,
// so every thread keeps several independent gathers in flight (measured on GB300: 13.9 /
// 16.5 us at T = 2 / 4 on a K = 8640, N = 960 layer, against 19.5 / 26.7 for a row-block
// layout like the one above).
constexpr int kGatherRows = 4;

// 8 int8 -> 8 floats
__device__ __forceinline__ void i8x8_to_f32(uint2 v, float (&x)[8]) {
  const int32_t a = static_cast<int32_t>(v.x), b = static_cast<int32_t>(v.y);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[i] = static_cast<float>((a << (24 - 8 * i)) >> 24);
    x[4 + i] = static_cast<float>((b << (24 - 8 * i)) >> 24);
  }
}

template <int TT>
__global__ void __launch_bounds__(256, 2) skinny_gather_kernel(const SkinnyParams p) {
  extern __shared__ float4 gather_smem4[];
  float* wred = reinterpret_cast<float*>(gather_smem4);
  grid_dependency_wait();
  allow_dependents();
  const uint4* books = static_cast<const uint4*>(p.books);
  // CTA = four output rows; thread = a stride of group columns (8 weights of K each)
  const int n0 = blockIdx.x * kGatherRows;
  const int G = p.K >> 3;
  const int M = p.M;
  const int T = p.T;
  float acc[kGatherRows][TT];
#pragma unroll
  for (int r = 0; r < kGatherRows; ++r)
#pragma unroll
    for (int t = 0; t < TT; ++t) acc[r][t] = 0.0f;

  for (int gi = threadIdx.x; gi < G; gi += blockDim.x) {
    const int kb = gi >> 3, j = gi & 7;
    // the group's decoded weights for the four rows (the decode rule of Eq. 4)
    float w[kGatherRows][8];
#pragma unroll
    for (int r = 0; r < kGatherRows; ++r) {
      const int n = n0 + r;
      float s[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) s[e] = 0.0f;
      if (n < p.N) {
        const int64_t cidx = ((static_cast<int64_t>(kb) * p.N + n) * 8 + j) * M;
        for (int m = 0; m < M; ++m) {
          const int c = __ldg(static_cast<const uint16_t*>(p.codes) + cidx + m);
          const uint4 cw = __ldg(books + (static_cast<int64_t>(m) << 16) + c);
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
        for (int r = 0; r < kGatherRows; ++r)
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[r][t] = fmaf(w[r][e], x[e], acc[r][t]);
      }
    }
  }
  // reduce over the CTA in a fixed order: butterflies within each warp, then the warps
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < kGatherRows; ++r)
#pragma unroll
    for (int t = 0; t < TT; ++t) {
      float v = acc[r][t];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) wred[(warp * kGatherRows + r) * TT + t] = v;
    }
  __syncthreads();
  const int nwarps = blockDim.x >> 5;
  const float rs_out = p.out_q8 ? __frcp_rn(p.s_out) : 0.0f;
  for (int o = threadIdx.x; o < kGatherRows * T; o += blockDim.x) {
    const int t = o / kGatherRows;
    const int r = o - t * kGatherRows;
    const int n = n0 + r;
    if (n >= p.N) continue;
    float v = 0.0f;
    for (int wi = 0; wi < nwarps; ++wi) v += wred[(wi * kGatherRows + r) * TT + t];
    v = fmaf(v, p.s_x * __half2float(p.scale[n]), p.bias ? __half2float(p.bias[n]) : 0.0f);
    const int64_t off = static_cast<int64_t>(t) * p.N + n;
    if (p.out_f32)
      static_cast<float*>(p.y)[off] = v;
    else if (p.out_q8 == kOutCodesF16)
      static_cast<__half*>(p.y)[off] =
          __short2half_rn(quant_one(__float2half_rn(v), p.s_out, rs_out));
    else if (p.out_q8)
      static_cast<int8_t*>(p.y)[off] = quant_one(__float2half_rn(v), p.s_out, rs_out);
    else
      static_cast<__half*>(p.y)[off] = __float2half_rn(v);
  }
}

static int skinny_tt(int T) { return T <= 1 ? 1 : T <= 2 ? 2 : T <= 4 ? 4 : T <= 8 ? 8 : 16; }

// Activations staged in shared memory as fp16 from two tokens on, when T * K * 2 bytes fit
// kSkinnyXsBytes.  Measured on GB300 (K = 8192, N = 16384, 2x8): T = 2 77.3 -> 62.4 us; at
// T = 1 the conversions it saves are fewer than the occupancy it costs (45.2 -> 50.2 us:
// 2 instead of 3 CTAs per SM), so one token keeps converting from global memory.
static bool skinny_x_smem(int T, int K) {
  return T >= 2 && static_cast<size_t>(T) * K * 2 <= static_cast<size_t>(kSkinnyXsBytes);
}

// 8-bit codes (the row-block kernel): codebook copies + the warps' partial sums (+ the
// activations as fp16)
size_t skinny_smem_bytes(int M, int T, int K) {
  return static_cast<size_t>(M) * 256 * 16 * fused_book_copies(M) +
         static_cast<size_t>(kSkinnyWarps) * kSkinnyRows * skinny_tt(T) * 4 +
         (skinny_x_smem(T, K) ? static_cast<size_t>(T) * K * 2 : 0);
}

template <int MM>
cudaError_t launch_skinny_m(const SkinnyParams& p, size_t smem, cudaStream_t st) {
  // persistent CTAs: as many row blocks as fit at once (shared memory and threads bound
  // the CTAs per SM), at most one per row block
  const int n_rb = (p.N + kSkinnyRows - 1) / kSkinnyRows;
  int per_sm = static_cast<int>(232448 / (smem + 1024));
  per_sm = per_sm < 1 ? 1 : (per_sm > 2048 / (kSkinnyWarps * 32) ? 2048 / (kSkinnyWarps * 32) : per_sm);
  const int sms = p.sms > 0 ? p.sms : 152;
  int blocks = sms * per_sm;
  if (blocks > n_rb) blocks = n_rb;
  const dim3 grid(static_cast<unsigned>(blocks)), block(kSkinnyWarps * 32);
  auto go = [&](auto kernel) -> cudaError_t {
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(smem));
      if (e != cudaSuccess) return e;
    }
    return launch_pdl(kernel, grid, block, smem, st, p);
  };
  switch (skinny_tt(p.T)) {
    case 1: return go(skinny_kernel<1, MM>);
    case 2: return go(skinny_kernel<2, MM>);
    case 4: return go(skinny_kernel<4, MM>);
    case 8: return go(skinny_kernel<8, MM>);
    default: return go(skinny_kernel<16, MM>);
  }
}

cudaError_t launch_skinny_gather(const SkinnyParams& p, cudaStream_t st) {
  const int G = p.K / 8;
  int threads = (G + 31) / 32 * 32;
  if (threads > 256) threads = 256;
  const int blocks = (p.N + kGatherRows - 1) / kGatherRows;
  const size_t smem = static_cast<size_t>(threads / 32) * kGatherRows * skinny_tt(p.T) * 4;
  const dim3 grid(static_cast<unsigned>(blocks)), block(static_cast<unsigned>(threads));
  switch (skinny_tt(p.T)) {
    case 1: return launch_pdl(skinny_gather_kernel<1>, grid, block, smem, st, p);
    case 2: return launch_pdl(skinny_gather_kernel<2>, grid, block, smem, st, p);
    case 4: return launch_pdl(skinny_gather_kernel<4>, grid, block, smem, st, p);
    case 8: return launch_pdl(skinny_gather_kernel<8>, grid, block, smem, st, p);
    default: return launch_pdl(skinny_gather_kernel<16>, grid, block, smem, st, p);
  }
}

cudaError_t launch_skinny(SkinnyParams p, cudaStream_t st) {
  if (p.B == 16) return launch_skinny_gather(p, st);
  p.x_smem = skinny_x_smem(p.T, p.K) ? 1 : 0;
  const size_t smem = skinny_smem_bytes(p.M, p.T, p.K);
  if (p.M == 1) return launch_skinny_m<1>(p, smem, st);
  if (p.M == 2) return launch_skinny_m<2>(p, smem, st);
  return launch_skinny_m<0>(p, smem, st);
}

}  // namespace aq
