// aq_gemm.cu -- tcgen05 tensor-core contraction of the AQ x A8 layer.
//
// acc[t][n] = sum_k fp16(xq[t][k]) * W[n][k]   (fp32 in TMEM), then the fused
// epilogue y = acc * (s_x * scale[n]) + bias[n] (Sec. 3.1.1: the layer is the
// product Y = W X; for a convolution X is the im2col matrix, built here tap by
// tap from 4-D TMA boxes instead of being materialised).
//
// One CTA computes a 128 x BN output tile (optionally one K split of it):
//   warp 0      TMA producer: int8 activation box + fp16 weight box per stage
//   warp 1      TMEM allocator and single-thread tcgen05.mma issuer
//   warps 2..5  int8 -> fp16 converters (into the 128B-swizzled K-major A
//               tile), then the epilogue (TMEM -> registers -> global)
// Stages are handed over with mbarriers; every wait is bounded (about 2 s),
// after which the CTA records an error, drains its own copies and exits.
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"

namespace aq {

__device__ unsigned g_gemm_err = 0;

constexpr int kStages = 3;
constexpr int kA16Bytes = kBM * 128;       // 16 KB fp16 A stage (128 rows x 64 fp16)
constexpr int kB16Bytes = kMaxBN * 128;    // 32 KB fp16 B stage (<= 256 rows x 64 fp16)
constexpr int kA8Bytes = kBM * 64;         // 8 KB int8 A stage
constexpr int kTmemCols = 256;

struct alignas(8) GemmSmemTail {
  uint64_t full[kStages];    // TMA bytes landed (A int8 + B fp16)
  uint64_t conv[kStages];    // A converted to fp16 (4 converter warps arrive)
  uint64_t empty[kStages];   // MMA finished reading the stage (tcgen05.commit)
  uint64_t accum;            // all MMAs of the tile done
  uint32_t tmem_base;
  int abort_flag;
  float scale[kMaxBN];       // s_x * scale[n]
  float bias[kMaxBN];
};

constexpr size_t kGemmSmemBytes =
    1024 /*alignment slack*/ + static_cast<size_t>(kStages) * (kA16Bytes + kB16Bytes + kA8Bytes) +
    sizeof(GemmSmemTail);

__device__ __forceinline__ void record_failure(GemmSmemTail* tl, unsigned code) {
  *reinterpret_cast<volatile int*>(&tl->abort_flag) = 1;
  atomicOr(&g_gemm_err, code);
}

__global__ void __launch_bounds__(192, 1)
    aq_gemm_kernel(const __grid_constant__ CUtensorMap mapA,
                   const __grid_constant__ CUtensorMap mapB, const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* a16 = smem;
  uint8_t* b16 = a16 + kStages * kA16Bytes;
  uint8_t* a8 = b16 + kStages * kB16Bytes;
  GemmSmemTail* tl = reinterpret_cast<GemmSmemTail*>(a8 + kStages * kA8Bytes);
  const volatile int* abort_flag = &tl->abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int BN = p.BN;
  const int n0 = blockIdx.x * BN;
  const int mt = blockIdx.y;
  const int m0 = mt * kBM;
  const int split = blockIdx.z;
  const int kb_begin = split * p.kb_per_split;
  const int kb_end = min(p.num_kb, kb_begin + p.kb_per_split);
  const int nk = kb_end - kb_begin;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&tl->full[s], 1);
      mbar_init(&tl->conv[s], 4);
      mbar_init(&tl->empty[s], 1);
    }
    mbar_init(&tl->accum, 1);
    tl->abort_flag = 0;
    mbar_fence_init();
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
  }
  if (warp == 1) {
    tmem_alloc(&tl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  for (int i = threadIdx.x; i < BN; i += blockDim.x) {
    const int n = n0 + i;
    tl->scale[i] = (n < p.N) ? p.s_x * __half2float(p.scale[n]) : 0.0f;
    tl->bias[i] = (n < p.N && p.bias != nullptr) ? __half2float(p.bias[n]) : 0.0f;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = tl->tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0 && nk > 0) {
      int b0 = 0, ho0 = 0;
      if (p.conv) {
        if (p.imgs_per_tile > 0) {
          b0 = mt * p.imgs_per_tile;
        } else {
          b0 = mt / p.tiles_per_img;
          ho0 = (mt % p.tiles_per_img) * p.rows_per_tile;
        }
      }
      const uint32_t stage_bytes = kA8Bytes + static_cast<uint32_t>(BN) * 128u;
      int issued = 0;
      for (int i = 0; i < nk; ++i) {
        const int s = i % kStages;
        const uint32_t ph = (i / kStages) & 1u;
        if (i >= kStages && !mbar_wait(&tl->empty[s], ph ^ 1u, abort_flag)) {
          record_failure(tl, kDevErrTimeoutEmpty);
          break;
        }
        if (*abort_flag) break;
        const int kb = kb_begin + i;
        mbar_arrive_expect_tx(&tl->full[s], stage_bytes);
        if (!p.conv) {
          tma_load_2d(a8 + s * kA8Bytes, &mapA, &tl->full[s], kb * kBK, m0);
        } else {
          const int tap = kb / p.cin_blocks;
          const int c0 = (kb - tap * p.cin_blocks) * kBK;
          const int kh = tap / 3, kw = tap - 3 * (tap / 3);
          tma_load_4d(a8 + s * kA8Bytes, &mapA, &tl->full[s], c0, kw - p.pad, ho0 + kh - p.pad,
                      b0);
        }
        tma_load_2d(b16 + s * kB16Bytes, &mapB, &tl->full[s], kb * kBK, n0);
        ++issued;
      }
      if (*abort_flag) {
        // drain: the last (up to kStages) issued stages may still be in flight
        const int zero = 0;
        for (int i = max(0, issued - kStages); i < issued; ++i) {
          if (!mbar_wait(&tl->full[i % kStages], (i / kStages) & 1u, &zero)) {
            atomicOr(&g_gemm_err, kDevErrTimeoutDrain);
            break;
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && nk > 0) {
      const uint32_t idesc = idesc_f16_f32(kBM, BN);
      for (int i = 0; i < nk; ++i) {
        const int s = i % kStages;
        const uint32_t ph = (i / kStages) & 1u;
        if (!mbar_wait(&tl->full[s], ph, abort_flag) || !mbar_wait(&tl->conv[s], ph, abort_flag)) {
          record_failure(tl, kDevErrTimeoutConv);
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_u32(a16 + s * kA16Bytes);
        const uint32_t b_base = smem_u32(b16 + s * kB16Bytes);
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k) {
          mma_f16_ss(tmem_base, sw128_kmajor_desc(a_base + 32u * k),
                     sw128_kmajor_desc(b_base + 32u * k), idesc, (i | k) != 0 ? 1u : 0u);
        }
        mma_commit(&tl->empty[s]);
      }
      mma_commit(&tl->accum);
      if (*abort_flag) {
        const int zero = 0;
        if (!mbar_wait(&tl->accum, 0, &zero)) atomicOr(&g_gemm_err, kDevErrTimeoutDrain);
      }
    }
  } else {
    // ------------------------------------------------------------ converters
    const int ct = threadIdx.x - 64;  // 0..127
    for (int i = 0; i < nk; ++i) {
      const int s = i % kStages;
      const uint32_t ph = (i / kStages) & 1u;
      if (!mbar_wait(&tl->full[s], ph, abort_flag)) {
        record_failure(tl, kDevErrTimeoutFull);
        break;
      }
      const uint8_t* src = a8 + s * kA8Bytes;
      uint8_t* dst = a16 + s * kA16Bytes;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int q = ct + 128 * j;
        const int row = q >> 2;
        const int c = q & 3;
        const uint4 v = *reinterpret_cast<const uint4*>(src + row * 64 + c * 16);
        uint32_t o[8];
        i8x4_to_f16x4(v.x, o[0], o[1]);
        i8x4_to_f16x4(v.y, o[2], o[3]);
        i8x4_to_f16x4(v.z, o[4], o[5]);
        i8x4_to_f16x4(v.w, o[6], o[7]);
        const int sw = row & 7;
        *reinterpret_cast<uint4*>(dst + row * 128 + (((2 * c) ^ sw) << 4)) =
            make_uint4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<uint4*>(dst + row * 128 + (((2 * c + 1) ^ sw) << 4)) =
            make_uint4(o[4], o[5], o[6], o[7]);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tl->conv[s]);
    }

    // ------------------------------------------------------------ epilogue
    bool ok = nk > 0 && mbar_wait(&tl->accum, 0, abort_flag);
    if (nk > 0 && !ok && !*abort_flag) record_failure(tl, kDevErrTimeoutAccum);
    ok = __all_sync(0xffffffffu, ok ? 1 : 0) != 0;
    if (ok) {
      tc_fence_after();
      const int qd = warp & 3;                 // TMEM lane quadrant of this warp
      const int row = qd * 32 + lane;
      const int t = m0 + row;
      const uint32_t tq = tmem_base + (static_cast<uint32_t>(qd * 32) << 16);
      const int cols = min(BN, p.N - n0);      // valid columns of this tile
      for (int c0 = 0; c0 < BN; c0 += 32) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tq + static_cast<uint32_t>(c0), r);
        tmem_wait_ld();
        if (t < p.T) {
          if (p.partial != nullptr) {
            float* dst = p.partial + (static_cast<int64_t>(split) * p.T + t) * p.N + n0;
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              if (c0 + j < cols)
                *reinterpret_cast<float4*>(dst + c0 + j) =
                    make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
            }
          } else if (p.out_f32) {
            float* dst = static_cast<float*>(p.y) + static_cast<int64_t>(t) * p.N + n0;
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
              if (c0 + j < cols) {
                float4 v;
                v.x = fmaf(__uint_as_float(r[j]), tl->scale[c0 + j], tl->bias[c0 + j]);
                v.y = fmaf(__uint_as_float(r[j + 1]), tl->scale[c0 + j + 1], tl->bias[c0 + j + 1]);
                v.z = fmaf(__uint_as_float(r[j + 2]), tl->scale[c0 + j + 2], tl->bias[c0 + j + 2]);
                v.w = fmaf(__uint_as_float(r[j + 3]), tl->scale[c0 + j + 3], tl->bias[c0 + j + 3]);
                *reinterpret_cast<float4*>(dst + c0 + j) = v;
              }
            }
          } else {
            __half* dst = static_cast<__half*>(p.y) + static_cast<int64_t>(t) * p.N + n0;
#pragma unroll
            for (int j = 0; j < 32; j += 8) {
              if (c0 + j < cols) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int cc = c0 + j + 2 * e;
                  const float lo = fmaf(__uint_as_float(r[j + 2 * e]), tl->scale[cc], tl->bias[cc]);
                  const float hi =
                      fmaf(__uint_as_float(r[j + 2 * e + 1]), tl->scale[cc + 1], tl->bias[cc + 1]);
                  __half2 h = __floats2half2_rn(lo, hi);
                  w[e] = *reinterpret_cast<uint32_t*>(&h);
                }
                *reinterpret_cast<uint4*>(dst + c0 + j) = make_uint4(w[0], w[1], w[2], w[3]);
              }
            }
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Sum of the split-K partials, then the fused epilogue.  One thread per 4 outputs.
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const GemmParams p, int splits) {
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < nq;
       q += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = q / (p.N / 4);
    const int n = static_cast<int>(q - t * (p.N / 4)) * 4;
    float4 acc = *reinterpret_cast<const float4*>(p.partial + t * p.N + n);
    for (int s = 1; s < splits; ++s) {
      const float4 v =
          *reinterpret_cast<const float4*>(p.partial + (static_cast<int64_t>(s) * p.T + t) * p.N + n);
      acc.x += v.x;
      acc.y += v.y;
      acc.z += v.z;
      acc.w += v.w;
    }
    float o[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float sc = p.s_x * __half2float(p.scale[n + e]);
      const float bi = p.bias ? __half2float(p.bias[n + e]) : 0.0f;
      o[e] = fmaf(o[e], sc, bi);
    }
    if (p.out_f32) {
      *reinterpret_cast<float4*>(static_cast<float*>(p.y) + t * p.N + n) =
          make_float4(o[0], o[1], o[2], o[3]);
    } else {
      __half2 a = __floats2half2_rn(o[0], o[1]);
      __half2 b = __floats2half2_rn(o[2], o[3]);
      uint2 w = make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
      *reinterpret_cast<uint2*>(static_cast<__half*>(p.y) + t * p.N + n) = w;
    }
  }
}

cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, const GemmParams& p,
                        int n_tiles, int m_tiles, int splits, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(aq_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kGemmSmemBytes));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid(n_tiles, m_tiles, splits);
  aq_gemm_kernel<<<grid, 192, kGemmSmemBytes, st>>>(mapA, mapB, p);
  return cudaGetLastError();
}

cudaError_t launch_splitk_reduce(const GemmParams& p, int splits, cudaStream_t st) {
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  int64_t blocks = (nq + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  splitk_reduce_kernel<<<static_cast<unsigned>(blocks), 256, 0, st>>>(p, splits);
  return cudaGetLastError();
}

cudaError_t read_clear_gemm_error(unsigned* out) {
  unsigned v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(v));
  if (e != cudaSuccess) return e;
  const unsigned zero = 0;
  e = cudaMemcpyToSymbol(g_gemm_err, &zero, sizeof(zero));
  *out = v;
  return e;
}

}  // namespace aq
