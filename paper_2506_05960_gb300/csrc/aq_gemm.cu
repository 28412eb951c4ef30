// aq_gemm.cu -- tcgen05 tensor-core contraction of the AQ x A8 layer.
//
// acc[t][n] = sum_k fp16(xq[t][k]) * W[n][k]   (fp32 in tensor memory), then the
// fused epilogue y = acc * (s_x * scale[n]) + bias[n] (Sec. 3.1.1: the layer is
// the product Y = W X; for a convolution X is the im2col matrix, assembled here
// from 4-D TMA boxes per (tap, 64-channel block) instead of being materialised).
//
// Persistent kernel, one CTA per SM, static round-robin over 128 x BN output
// tiles (and K splits).  A pipeline stage covers 128 of K (two 64-wide TMA
// boxes per operand, eight 128 x BN x 16 MMAs).  Ten warps, fourteen on the dense path
// with 8 epilogue warps, sixteen on the fused path:
//   warp 0      TMA producer: int8 activation boxes (64-byte swizzle) and fp16
//               weight boxes (128-byte swizzle) into an S-deep smem ring
//   warp 1      TMEM owner (all 512 columns) and the single MMA-issuing thread:
//               tcgen05.mma.kind::f16 with A read from TMEM and B from shared
//               memory.  Its loop is kept minimal (one barrier wait per eight
//               MMAs, descriptors advanced by addition, no divisions): with
//               BN = 192 the wait, fence and commits hide under the MMAs.
//   warps 2..5  converters: int8 rows -> fp16 exactly -> tcgen05.st into a
//               TMEM A ring (no shared-memory round trip for the fp16 operand)
//   warps 6..9  epilogue: TMEM accumulator -> scale/bias -> 32 x 32 boxes in
//   (6..13)     shared memory -> TMA stores (ragged edges clipped by TMA).  The
//               output is fp16, fp32, or int8: the fp16 value quantized with the
//               next layer's activation scale (the quantizer fused into the layer).
//               A warp reads only its TMEM lane quarter (warp % 4), so 8 epilogue
//               warps pair up per quarter and take alternate 32-column chunks: with
//               small K the epilogue, not the mainloop, bounds a tile.
//   warps 10..15 (fused path) decoders: rebuild each weight stage from the packed
//               codes and the shared-memory codebooks (Eq. 4).  The lookups are
//               bound by shared-memory bandwidth, hence six warps and the
//               bank-spread codebook copies (fused_book_copies).
// The fp32 accumulator is double-buffered in TMEM so the epilogue of one tile
// runs under the mainloop of the next.  The issue loop carries no divisions:
// ring index and phase advance by counters.  Every wait is bounded (about 2 s);
// on time-out the CTA records an error word, drains its in-flight work, frees
// TMEM and exits.
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "aq_internal.h"
#include "aq_ptx.cuh"
#include "aq_quant.cuh"

namespace aq {

__device__ unsigned g_gemm_err = 0;

constexpr int kDecodeThreads = 192;             // warps 10..15 decode on the fused path
constexpr int kThreads = 320 + kDecodeThreads;
constexpr int kA8Half = kBM * 64;               // one 64-wide int8 box: 128 rows x 64 B
constexpr int kA8Stage = kStageBlocks * kA8Half;
constexpr int kA16Half = kBM * 128;             // one 64-wide fp16 A box: 128 rows x 128 B
constexpr int kASlotCols = kStageBlocks * 32;   // TMEM columns of one fp16 A slot
constexpr int kEpiBuf32 = 4096;                 // one 32 x 32 fp32 output box (128-byte rows)
constexpr int kEpiBuf16 = 2048;                 // one 32 x 32 fp16 output box (64-byte rows)
// Epilogue staging per warp: 4 warps keep two output boxes and the scale/bias of all BN
// columns each; 8 or 12 warps (two or three per lane quarter, taking its 32-column chunks in
// turn) keep one box and the scale/bias of their own columns.
__host__ __device__ constexpr int epi_out_bufs(int epi_warps) { return epi_warps >= 8 ? 1 : 2; }
// Columns of scale/bias a warp keeps: its 32-column chunks of a BN-wide tile, compacted.
__host__ __device__ constexpr int epi_scale_cols(int epi_warps, int BN) {
  return ((BN + 31) / 32 + epi_warps / 4 - 1) / (epi_warps / 4) * 32;
}
// Bytes of A per pipeline stage: int8 boxes (TMEM-A form) or fp16 boxes (shared-memory A).
__host__ __device__ constexpr int a_stage_bytes(bool a16, int sb) {
  return a16 ? sb * kA16Half : kA8Stage;
}
constexpr int kTmemCols = 512;

struct alignas(8) GemmBarriers {
  uint64_t full[kMaxStages];     // TMA bytes of a smem stage landed
  uint64_t empty[kMaxStages];    // smem stage consumed: 4 converter warps + 1 MMA commit
                                 // (shared-memory A form: the MMA commit alone)
  uint32_t a_ready[kMaxStages];  // fp16 A slot written: +1 per converter warp (4 per use)
  uint64_t a_empty[kMaxStages];  // MMAs reading the TMEM slot done (commit)
  uint64_t acc_full[2];          // accumulator buffer complete (commit)
  uint64_t acc_empty[2];         // accumulator buffer drained (one arrival per epilogue warp)
  uint64_t drain;                // all MMAs of this CTA complete (teardown)
  uint64_t codes_full[kMaxStages];  // fused path: a stage's packed codes landed in smem
  uint32_t tmem_base;
  int abort_flag;
};

// code_bytes: packed code bytes of one row for one 64-wide K block on the fused path
// (8 * M * bytes per code), 0 on the dense path.
size_t gemm_smem_bytes(int BN, int stages, bool f32_out, int book_bytes, int code_bytes,
                       int epi_warps, bool a16, int sb) {
  const int SB = a16 ? sb : kStageBlocks;
  return 1024 +
         static_cast<size_t>(stages) *
             (SB * BN * 128 + a_stage_bytes(a16, sb) + SB * BN * code_bytes) +
         static_cast<size_t>(epi_warps) * (epi_out_bufs(epi_warps) * (f32_out ? kEpiBuf32 : kEpiBuf16) +
                                           2 * epi_scale_cols(epi_warps, BN) * 4) +
         book_bytes + sizeof(GemmBarriers);
}

int gemm_max_stages(int BN, bool f32_out, int book_bytes, int code_bytes, int epi_warps,
                    bool a16, int sb) {
  const size_t fixed = gemm_smem_bytes(BN, 0, f32_out, book_bytes, code_bytes, epi_warps, a16, sb);
  const int SB = a16 ? sb : kStageBlocks;
  const size_t per = static_cast<size_t>(SB) * BN * (128 + code_bytes) + a_stage_bytes(a16, sb);
  const int s = static_cast<int>((232448 - fixed) / per);
  return s < kMaxStages ? s : kMaxStages;
}

int gemm_a_stages(int BN) {
  const int s = (kTmemCols - 2 * BN) / kASlotCols;
  return s < kMaxStages ? s : kMaxStages;
}

__device__ __forceinline__ void record_failure(GemmBarriers* b, unsigned code) {
  *reinterpret_cast<volatile int*>(&b->abort_flag) = 1;
  atomicOr(&g_gemm_err, code);
}

struct TileCoord {
  int m_tile, n_tile, split, kb_begin, kb_end;
};

__device__ __forceinline__ TileCoord tile_coord(const GemmParams& p, int t) {
  TileCoord c;
  int r;
  if (p.cluster) {
    // the splits of one tile are consecutive CTAs: one cluster
    r = t / p.splits;
    c.split = t - r * p.splits;
  } else {
    const int tiles_mn = p.m_tiles * p.n_tiles;
    c.split = t / tiles_mn;
    r = t - c.split * tiles_mn;
  }
  c.n_tile = r / p.m_tiles;
  c.m_tile = r - c.n_tile * p.m_tiles;
  c.kb_begin = c.split * p.kb_per_split;
  c.kb_end = min(p.num_kb, c.kb_begin + p.kb_per_split);
  return c;
}

// N of the tile's MMAs: its valid output columns rounded up to 16 (the instruction's
// granularity for M = 128); columns past them are never stored.
__device__ __forceinline__ int tile_mma_n(const GemmParams& p, const TileCoord& tc) {
  const int valid = p.N - tc.n_tile * p.BN;
  return valid >= p.BN ? p.BN : ((valid + 15) & ~15);
}

// Ring position: slot index and the parity of the slot's current lap.
struct Ring {
  int s = 0;
  uint32_t ph = 0;
  uint32_t lap0 = 1;  // 1 while still in the first lap over the slots
  __device__ __forceinline__ void next(int S) {
    if (++s == S) {
      s = 0;
      ph ^= 1u;
      lap0 = 0;
    }
  }
};

// Sum of the M codewords of one group in fp32 (ascending m), one RNE to fp16 (Eq. 4).
// For M <= 2 the fp16 adds give the same bits: the exact sum of two fp16 values
// rounded once to fp32 and then to fp16 equals its direct fp16 rounding, since
// fp32 carries at least 2 * 11 + 2 significand bits (double rounding is innocuous).
template <int M>
__device__ __forceinline__ uint4 sum_codewords(const uint4* word) {
  if constexpr (M == 1) {
    return word[0];
  } else if constexpr (M == 2) {
    uint4 out;
    const __half2* a = reinterpret_cast<const __half2*>(&word[0]);
    const __half2* b = reinterpret_cast<const __half2*>(&word[1]);
    __half2* o = reinterpret_cast<__half2*>(&out);
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = __hadd2(a[i], b[i]);
    return out;
  } else {
    float acc[8];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      const __half2* h2 = reinterpret_cast<const __half2*>(&word[m]);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(h2[i]);
        acc[2 * i] = m == 0 ? f.x : __fadd_rn(acc[2 * i], f.x);
        acc[2 * i + 1] = m == 0 ? f.y : __fadd_rn(acc[2 * i + 1], f.y);
      }
    }
    uint4 out;
    uint32_t* o = reinterpret_cast<uint32_t*>(&out);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __half2 hh = __floats2half2_rn(acc[2 * i], acc[2 * i + 1]);
      o[i] = *reinterpret_cast<uint32_t*>(&hh);
    }
    return out;
  }
}

// Fused path: decode the 8 groups of one output row in one 64-wide K block into the
// row's 128-byte line of the swizzled B stage.  Codes: 8*M*EB contiguous bytes in
// shared memory (EB = bytes per code), read as 32-bit words and unpacked with
// constant shifts.  8-bit codes index the codebooks staged in shared memory (this
// lane's copy `copy` of fused_book_copies(M)); 16-bit codes gather from L2, all 8*M
// reads issued before the first sum.
template <int M, int EB>
__device__ __forceinline__ void decode_unit(const uint8_t* codes, const uint4* sbook,
                                            const uint4* gbooks, uint8_t* rowp, int n,
                                            int gvalid, int copy) {
  constexpr int R = fused_book_copies(M);
  constexpr int kWords = 2 * M * EB;
  uint32_t w[kWords];
  if constexpr (kWords % 4 == 0) {
#pragma unroll
    for (int i = 0; i < kWords / 4; ++i) {
      const uint4 v = reinterpret_cast<const uint4*>(codes)[i];
      w[4 * i] = v.x;
      w[4 * i + 1] = v.y;
      w[4 * i + 2] = v.z;
      w[4 * i + 3] = v.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < kWords / 2; ++i) {
      const uint2 v = reinterpret_cast<const uint2*>(codes)[i];
      w[2 * i] = v.x;
      w[2 * i + 1] = v.y;
    }
  }
  constexpr int kPre = EB == 2 ? 8 * M : 1;
  uint4 cw[kPre];
  if (EB == 2) {
#pragma unroll
    for (int idx = 0; idx < 8 * M; ++idx) {
      const uint32_t c = (w[idx >> 1] >> (16 * (idx & 1))) & 0xFFFFu;
      const int m = idx % M;
      cw[idx % kPre] = (idx / M) < gvalid ? __ldg(gbooks + (static_cast<int64_t>(m) << 16) + c)
                                          : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  if constexpr (EB == 1) {
    // the codewords of J groups are loaded before any of them is stored: loads and
    // stores share no ordering the compiler can prove, so a per-group loop would
    // serialise every lookup behind the previous store (codes past gvalid are zero
    // bytes in the packed layout, so their lookups stay inside the table)
    constexpr int J = M <= 2 ? 4 : (M <= 4 ? 2 : 1);
#pragma unroll
    for (int j0 = 0; j0 < 8; j0 += J) {
      uint4 word[J * M];
#pragma unroll
      for (int i = 0; i < J * M; ++i) {
        const int idx = j0 * M + i;
        word[i] = sbook[((i % M) * 256 + ((w[idx >> 2] >> (8 * (idx & 3))) & 0xFFu)) * R + copy];
      }
#pragma unroll
      for (int jj = 0; jj < J; ++jj) {
        const int j = j0 + jj;
        uint4 out = sum_codewords<M>(word + jj * M);
        if (j >= gvalid) out = make_uint4(0u, 0u, 0u, 0u);
        *reinterpret_cast<uint4*>(rowp + ((j ^ (n & 7)) << 4)) = out;
      }
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const uint4 out = j < gvalid ? sum_codewords<M>(cw + j * M) : make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(rowp + ((j ^ (n & 7)) << 4)) = out;
    }
  }
}

__device__ __forceinline__ void decode_unit_dispatch(int M, int EB, const uint8_t* codes,
                                                     const uint4* sbook, const uint4* gbooks,
                                                     uint8_t* rowp, int n, int gvalid,
                                                     int copy) {
  if (EB == 1) {
    switch (M) {
      case 1: decode_unit<1, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 2: decode_unit<2, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 3: decode_unit<3, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 4: decode_unit<4, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 5: decode_unit<5, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 6: decode_unit<6, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      case 7: decode_unit<7, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
      default: decode_unit<8, 1>(codes, sbook, gbooks, rowp, n, gvalid, copy); break;
    }
  } else {
    if (M == 1)
      decode_unit<1, 2>(codes, sbook, gbooks, rowp, n, gvalid, copy);
    else
      decode_unit<2, 2>(codes, sbook, gbooks, rowp, n, gvalid, copy);
  }
}

// Epilogue of four summed split-K outputs y[t][n .. n+3]: acc * (s_x * scale) + bias in
// fp32, then fp32, fp16 or the 8-bit activation rule (the same arithmetic as the
// single-pass epilogue).
// s_x * scale and bias of output columns n .. n+3 (n % 4 == 0: one 8-byte load each).
__device__ __forceinline__ void load_scale_bias4(const GemmParams& p, int n, float (&sc)[4],
                                                 float (&bi)[4]) {
  const uint2 s2 = *reinterpret_cast<const uint2*>(p.scale + n);
  const uint2 b2 = p.bias ? *reinterpret_cast<const uint2*>(p.bias + n) : make_uint2(0u, 0u);
  const __half2 s01 = *reinterpret_cast<const __half2*>(&s2.x);
  const __half2 s23 = *reinterpret_cast<const __half2*>(&s2.y);
  const __half2 b01 = *reinterpret_cast<const __half2*>(&b2.x);
  const __half2 b23 = *reinterpret_cast<const __half2*>(&b2.y);
  sc[0] = p.s_x * __low2float(s01);
  sc[1] = p.s_x * __high2float(s01);
  sc[2] = p.s_x * __low2float(s23);
  sc[3] = p.s_x * __high2float(s23);
  bi[0] = __low2float(b01);
  bi[1] = __high2float(b01);
  bi[2] = __low2float(b23);
  bi[3] = __high2float(b23);
}

// The epilogue of four consecutive outputs with their scale and bias given.
__device__ __forceinline__ void store_out4_sb(const GemmParams& p, int64_t t, int n, float4 acc,
                                              const float (&sc)[4], const float (&bi)[4]) {
  float o[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
  for (int e = 0; e < 4; ++e) o[e] = fmaf(o[e], sc[e], bi[e]);
  if (p.out_f32) {
    *reinterpret_cast<float4*>(static_cast<float*>(p.y) + t * p.N + n) =
        make_float4(o[0], o[1], o[2], o[3]);
  } else if (p.out_q8) {
    const float rs = __frcp_rn(p.s_out);
    uint32_t b = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e)
      b |= static_cast<uint32_t>(static_cast<uint8_t>(quant_one(__float2half_rn(o[e]), p.s_out, rs)))
           << (8 * e);
    if (p.out_q8 == kOutCodesF16) {
      uint32_t lo, hi;
      i8x4_to_f16x4(b, lo, hi);
      *reinterpret_cast<uint2*>(static_cast<__half*>(p.y) + t * p.N + n) = make_uint2(lo, hi);
    } else {
      *reinterpret_cast<uint32_t*>(static_cast<int8_t*>(p.y) + t * p.N + n) = b;
    }
  } else {
    __half2 a = __floats2half2_rn(o[0], o[1]);
    __half2 b = __floats2half2_rn(o[2], o[3]);
    uint2 w = make_uint2(*reinterpret_cast<uint32_t*>(&a), *reinterpret_cast<uint32_t*>(&b));
    *reinterpret_cast<uint2*>(static_cast<__half*>(p.y) + t * p.N + n) = w;
  }
}

__device__ __forceinline__ void store_out4(const GemmParams& p, int64_t t, int n, float4 acc) {
  float sc[4], bi[4];
  load_scale_bias4(p, n, sc, bi);
  store_out4_sb(p, t, n, acc, sc, bi);
}

// kA16: the shared-memory A form (GemmParams::a16): fp16 A boxes with the 128-byte swizzle
// beside the weight boxes, tcgen05.mma with both operands from shared memory, no converter
// warps; warps 2.. are the epilogue and the TMEM holds only the two accumulators (BN <= 256).
template <bool kA16>
__global__ void __launch_bounds__(kThreads, 1)
    aq_gemm_kernel(const __grid_constant__ CUtensorMap mapA,
                   const __grid_constant__ CUtensorMap mapB,
                   const __grid_constant__ CUtensorMap mapY, const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  const int SA = p.a_stages;
  const int BN = p.BN;
  const int SB = kA16 ? p.sb : kStageBlocks;  // 64-wide K blocks per stage
  const int a_half = kA16 ? kA16Half : kA8Half;  // one 64-wide A box
  const int a_stage = a_stage_bytes(kA16, SB);
  const int b_half = BN * 128;                 // one 64-wide fp16 B box
  const int b_stage = SB * b_half;
  const bool raw = p.partial != nullptr;
  const bool f32 = raw || p.out_f32;
  const int epi_buf = f32 ? kEpiBuf32 : kEpiBuf16;
  uint8_t* bring = smem;
  uint8_t* aring = bring + S * b_stage;
  uint8_t* epi = aring + S * a_stage;
  const int EW = p.epi_warps;                  // 4, 8 or 12 (1-3 per TMEM lane quarter)
  const int epi_first = kA16 ? 2 : 6;          // first epilogue warp
  float* sscale = reinterpret_cast<float*>(epi + EW * epi_out_bufs(EW) * epi_buf);
  uint4* sbook = reinterpret_cast<uint4*>(reinterpret_cast<uint8_t*>(sscale) +
                                          EW * 2 * epi_scale_cols(EW, BN) * 4);
  // fused path: each stage's packed codes, [h][BN rows][code_bytes] (16-byte aligned)
  const int code_bytes = p.fused ? 8 * p.M * (p.B >> 3) : 0;
  const int code_stage = kStageBlocks * BN * code_bytes;
  uint8_t* scodes = reinterpret_cast<uint8_t*>(sbook) + p.book_bytes;
  GemmBarriers* bar = reinterpret_cast<GemmBarriers*>(scodes + S * code_stage);
  const volatile int* abort_flag = &bar->abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  // Barriers and tensor memory are set up while the previous kernel in the stream may
  // still run (programmatic launch); nothing in global memory is touched before it is done.
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      // fused path: the producer's expect_tx arrival + one arrival per decoder warp
      mbar_init(&bar->full[s], p.fused ? 1 + kDecodeThreads / 32 : 1);
      // fp16 A form: the MMA commit alone
      mbar_init(&bar->empty[s], kA16 ? 1 : 5);
    }
    for (int s = 0; s < SA; ++s) {
      bar->a_ready[s] = 0;
      mbar_init(&bar->a_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&bar->acc_full[b], 1);
      mbar_init(&bar->acc_empty[b], EW);
    }
    mbar_init(&bar->drain, 1);
    for (int s = 0; s < S; ++s) mbar_init(&bar->codes_full[s], 1);
    bar->abort_flag = 0;
    mbar_fence_init();
    tma_prefetch_desc(&mapA);
    if (!p.fused) tma_prefetch_desc(&mapB);
    tma_prefetch_desc(&mapY);
    if (p.fused && blockIdx.x < p.total_tiles) {
      // the weights do not come from the previous kernel: their first stages (and the
      // 8-bit codebooks) start moving into L2 while it still runs
      const TileCoord tc = tile_coord(p, blockIdx.x);
      const int n0 = tc.n_tile * BN;
      const int rows = min(BN, p.N - n0);
      const int cb = 8 * p.M * (p.B >> 3);
      const int kb_last = min(tc.kb_end, tc.kb_begin + kStageBlocks * S);
      for (int kb = tc.kb_begin; kb < kb_last; ++kb)
        bulk_prefetch_l2(static_cast<const uint8_t*>(p.codes) +
                             (static_cast<int64_t>(kb) * p.N + n0) * cb,
                         static_cast<uint32_t>(rows * cb));
      if (p.book_bytes > 0) bulk_prefetch_l2(p.books, static_cast<uint32_t>(p.M * 256 * 16));
    }
  }
  if (warp == 1) {
    tmem_alloc(&bar->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  grid_dependency_wait();
  allow_dependents();
  const uint32_t tmem_base = bar->tmem_base;

  if (warp == 0) {
    // ================================================================ TMA producer
    if (lane == 0) {
      Ring rg;
      uint32_t issued = 0;
      bool failed = false;
      for (int t = blockIdx.x; t < p.total_tiles && !failed; t += gridDim.x) {
        const TileCoord tc = tile_coord(p, t);
        const int m0 = tc.m_tile * kBM;
        const int n0 = tc.n_tile * BN;
        int b0 = 0, ho0 = 0, tap = 0, cb = 0;
        if (p.conv) {
          if (p.imgs_per_tile > 0) {
            b0 = tc.m_tile * p.imgs_per_tile;
          } else {
            b0 = tc.m_tile / p.tiles_per_img;
            ho0 = (tc.m_tile - b0 * p.tiles_per_img) * p.rows_per_tile;
          }
          tap = tc.kb_begin / p.cin_blocks;
          cb = tc.kb_begin - tap * p.cin_blocks;
        }
        for (int kb = tc.kb_begin; kb < tc.kb_end; kb += SB) {
          const int nb = min(SB, tc.kb_end - kb);
          if (!rg.lap0 && !mbar_wait(&bar->empty[rg.s], rg.ph ^ 1u, abort_flag, p.wait_ns)) {
            if (!*abort_flag) record_failure(bar, kDevErrTimeoutEmpty);
            failed = true;
            break;
          }
          uint64_t* fb = &bar->full[rg.s];
          if (p.fused) {
            // the stage's codes: per K block, rows n0 .. n0+rows-1 are contiguous in
            // the packed layout (rows is a multiple of 8, so sizes are multiples of 16)
            const int rows = min(BN, p.N - n0);
            const uint32_t bytes = static_cast<uint32_t>(rows * code_bytes);
            uint64_t* cbar = &bar->codes_full[rg.s];
            mbar_arrive_expect_tx(cbar, nb * bytes);
            for (int h = 0; h < nb; ++h)
              bulk_load(scodes + rg.s * code_stage + h * BN * code_bytes,
                        static_cast<const uint8_t*>(p.codes) +
                            (static_cast<int64_t>(kb + h) * p.N + n0) * code_bytes,
                        bytes, cbar);
          }
          mbar_arrive_expect_tx(fb, static_cast<uint32_t>(nb * (a_half + (p.fused ? 0 : b_half))));
          uint8_t* a_dst = aring + rg.s * a_stage;
          uint8_t* b_dst = bring + rg.s * b_stage;
          for (int h = 0; h < nb; ++h) {
            const int k = kb + h;
            if (!p.conv) {
              tma_load_2d(a_dst + h * a_half, &mapA, fb, k * kBK, m0);
            } else {
              const int kh = tap / 3, kw = tap - 3 * (tap / 3);
              tma_load_4d(a_dst + h * a_half, &mapA, fb, cb * kBK, kw - p.pad, ho0 * p.stride + kh - p.pad, b0);
              if (++cb == p.cin_blocks) {
                cb = 0;
                ++tap;
              }
            }
            if (!p.fused) tma_load_2d(b_dst + h * b_half, &mapB, fb, k * kBK, n0);
          }
          ++issued;
          rg.next(S);
        }
      }
      if (*abort_flag) {
        // drain: the stages issued in the last lap may still be in flight
        const int zero = 0;
        Ring d;
        const uint32_t first = issued > static_cast<uint32_t>(S) ? issued - S : 0u;
        for (uint32_t i = 0; i < issued; ++i) {
          if (i >= first && (!mbar_wait(&bar->full[d.s], d.ph, &zero) ||
                             (p.fused && !mbar_wait(&bar->codes_full[d.s], d.ph, &zero)))) {
            atomicOr(&g_gemm_err, kDevErrTimeoutDrain);
            break;
          }
          d.next(S);
        }
      }
    }
  } else if (warp == 1 && kA16) {
    // ================================================================ MMA issuer (A in smem)
    // Per stage: wait for its TMA bytes, four 128 x BN x 16 MMAs per 64-wide K block with
    // both operands read from the swizzled shared-memory boxes, one commit that frees the
    // stage for the producer.
    if (lane == 0) {
      const uint64_t adesc0 = sw128_kmajor_desc(smem_u32(aring));
      const uint64_t bdesc0 = sw128_kmajor_desc(smem_u32(bring));
      const uint64_t astep = static_cast<uint64_t>(a_stage >> 4);  // descriptor units: 16 B
      const uint64_t bstep = static_cast<uint64_t>(b_stage >> 4);
      const uint64_t ahalf = static_cast<uint64_t>(kA16Half >> 4);
      const uint64_t bhalf = static_cast<uint64_t>(b_half >> 4);
      Ring rg;
      uint32_t lt = 0;
      bool failed = false;
      for (int t = blockIdx.x; t < p.total_tiles && !failed; t += gridDim.x, ++lt) {
        const TileCoord tc = tile_coord(p, t);
        const int nblk = tc.kb_end - tc.kb_begin;
        // a ragged last N tile runs narrower MMAs (its valid columns, rounded up to 16)
        const uint32_t idesc = idesc_f16_f32(kBM, tile_mma_n(p, tc));
        const int buf = static_cast<int>(lt & 1u);
        if (lt >= 2 && !mbar_wait(&bar->acc_empty[buf], ((lt >> 1) & 1u) ^ 1u, abort_flag, p.wait_ns)) {
          if (!*abort_flag) record_failure(bar, kDevErrTimeoutAccum);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(buf * p.acc_stride);
        for (int kb = 0; kb < nblk; kb += SB) {
          const int nb = min(SB, nblk - kb);
          if (!mbar_wait(&bar->full[rg.s], rg.ph, abort_flag, p.wait_ns)) {
            if (!*abort_flag) record_failure(bar, kDevErrTimeoutFull);
            failed = true;
            break;
          }
          tc_fence_after();
          const uint64_t a0 = adesc0 + static_cast<uint64_t>(rg.s) * astep;
          const uint64_t b0 = bdesc0 + static_cast<uint64_t>(rg.s) * bstep;
          for (int h = 0; h < nb; ++h) {
            const uint64_t ah = a0 + static_cast<uint64_t>(h) * ahalf;
            const uint64_t bh = b0 + static_cast<uint64_t>(h) * bhalf;
            mma_f16_ss(d, ah, bh, idesc, (kb | h) ? 1u : 0u);
            mma_f16_ss(d, ah + 2u, bh + 2u, idesc, 1u);
            mma_f16_ss(d, ah + 4u, bh + 4u, idesc, 1u);
            mma_f16_ss(d, ah + 6u, bh + 6u, idesc, 1u);
          }
          mma_commit(&bar->empty[rg.s]);
          rg.next(S);
        }
        if (!failed) mma_commit(&bar->acc_full[buf]);
      }
      // every MMA of this CTA completes before teardown frees tensor memory
      mma_commit(&bar->drain);
      const int zero = 0;
      if (!mbar_wait(&bar->drain, 0, &zero)) atomicOr(&g_gemm_err, kDevErrTimeoutDrain);
    }
  } else if (warp == 1) {
    // ================================================================ MMA issuer
    if (lane == 0) {
      const uint64_t bdesc0 = sw128_kmajor_desc(smem_u32(bring));
      const uint64_t bstep = static_cast<uint64_t>(b_stage >> 4);  // descriptor units: 16 B
      const uint64_t bhalf = static_cast<uint64_t>(b_half >> 4);
      const uint32_t a_slot0 = tmem_base + static_cast<uint32_t>(p.a_col);
      int s = 0, sa = 0;
      uint32_t a_target = 4;     // a_ready value that marks the current lap of the A ring
      uint32_t lt = 0;
      bool failed = false;
      for (int t = blockIdx.x; t < p.total_tiles && !failed; t += gridDim.x, ++lt) {
        const TileCoord tc = tile_coord(p, t);
        const int nblk = tc.kb_end - tc.kb_begin;
        const uint32_t idesc = idesc_f16_f32(kBM, tile_mma_n(p, tc));
        const int nst = (nblk + 1) >> 1;
        const bool half_tail = (nblk & 1) != 0;
        const int buf = static_cast<int>(lt & 1u);
        if (lt >= 2 && !mbar_wait(&bar->acc_empty[buf], ((lt >> 1) & 1u) ^ 1u, abort_flag, p.wait_ns)) {
          if (!*abort_flag) record_failure(bar, kDevErrTimeoutAccum);
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(buf * p.acc_stride);
        for (int st = 0; st < nst; ++st) {
          if (!ctr_wait(&bar->a_ready[sa], a_target, abort_flag, p.wait_ns)) {
            if (!*abort_flag) record_failure(bar, kDevErrTimeoutConv);
            failed = true;
            break;
          }
          tc_fence_after();
          const uint32_t a = a_slot0 + static_cast<uint32_t>(kASlotCols * sa);
          const uint64_t b0 = bdesc0 + static_cast<uint64_t>(s) * bstep;
          const uint64_t b1 = b0 + bhalf;
          mma_f16_ts(d, a, b0, idesc, st > 0 ? 1u : 0u);
          mma_f16_ts(d, a + 8u, b0 + 2u, idesc, 1u);
          mma_f16_ts(d, a + 16u, b0 + 4u, idesc, 1u);
          mma_f16_ts(d, a + 24u, b0 + 6u, idesc, 1u);
          if (!(half_tail && st == nst - 1)) {
            mma_f16_ts(d, a + 32u, b1, idesc, 1u);
            mma_f16_ts(d, a + 40u, b1 + 2u, idesc, 1u);
            mma_f16_ts(d, a + 48u, b1 + 4u, idesc, 1u);
            mma_f16_ts(d, a + 56u, b1 + 6u, idesc, 1u);
          }
          mma_commit(&bar->empty[s]);
          mma_commit(&bar->a_empty[sa]);
          if (++s == S) s = 0;
          if (++sa == SA) {
            sa = 0;
            a_target += 4;
          }
        }
        if (!failed) mma_commit(&bar->acc_full[buf]);
      }
      // every MMA of this CTA completes before teardown frees tensor memory
      mma_commit(&bar->drain);
      const int zero = 0;
      if (!mbar_wait(&bar->drain, 0, &zero)) atomicOr(&g_gemm_err, kDevErrTimeoutDrain);
    }
  } else if (!kA16 && warp < 6) {
    // ================================================================ converters
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int swz = (row >> 1) & 3;            // 64-byte swizzle of the int8 box
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    Ring rg;   // smem ring
    Ring ra;   // TMEM A ring
    bool failed = false;
    for (int t = blockIdx.x; t < p.total_tiles && !failed; t += gridDim.x) {
      const TileCoord tc = tile_coord(p, t);
      for (int kb = tc.kb_begin; kb < tc.kb_end; kb += kStageBlocks) {
        const int nb = min(kStageBlocks, tc.kb_end - kb);
        bool okw = mbar_wait(&bar->full[rg.s], rg.ph, abort_flag, p.wait_ns);
        if (okw && !ra.lap0) okw = mbar_wait(&bar->a_empty[ra.s], ra.ph ^ 1u, abort_flag, p.wait_ns);
        if (!okw) {
          if (!*abort_flag) record_failure(bar, kDevErrTimeoutFull);
          failed = true;
          break;
        }
        tc_fence_after();
        const uint8_t* src = aring + rg.s * kA8Stage + row * 64;
        const uint32_t slot = t_row + static_cast<uint32_t>(p.a_col + kASlotCols * ra.s);
        for (int h = 0; h < nb; ++h) {
          uint32_t v[32];
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const uint4 w = *reinterpret_cast<const uint4*>(src + h * kA8Half + ((c ^ swz) << 4));
            i8x4_to_f16x4(w.x, v[8 * c + 0], v[8 * c + 1]);
            i8x4_to_f16x4(w.y, v[8 * c + 2], v[8 * c + 3]);
            i8x4_to_f16x4(w.z, v[8 * c + 4], v[8 * c + 5]);
            i8x4_to_f16x4(w.w, v[8 * c + 6], v[8 * c + 7]);
          }
          tmem_st_32x32b_x32(slot + 32u * h, v);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          smem_release_add(&bar->a_ready[ra.s], 1u);
          mbar_arrive(&bar->empty[rg.s]);
        }
        rg.next(S);
        ra.next(SA);
      }
    }
  } else if (warp < epi_first + EW) {
    // ================================================================ epilogue
    const int q = warp & 3;
    const int ew = warp - epi_first;
    // with 8 epilogue warps the two warps of a lane quarter take alternate 32-column chunks
    const int c_first = 32 * (ew >> 2);
    const int c_step = 32 * (EW >> 2);
    const int wcols = epi_scale_cols(EW, BN);  // this warp's chunks' columns, compacted
    const int nbuf = epi_out_bufs(EW);
    float* wscale = sscale + ew * 2 * wcols;
    float* wbias = wscale + wcols;
    uint8_t* wbuf = epi + ew * nbuf * epi_buf;
    const uint32_t t_row = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    const float rs_out = p.out_q8 ? __frcp_rn(p.s_out) : 0.0f;
    uint32_t lt = 0, chunk = 0;
    for (int t = blockIdx.x; t < p.total_tiles; t += gridDim.x, ++lt) {
      const TileCoord tc = tile_coord(p, t);
      const int buf = static_cast<int>(lt & 1u);
      const int m0 = tc.m_tile * kBM;
      const int n0 = tc.n_tile * BN;
      if (!raw && !p.cluster) {
        // this tile's scale/bias, loaded while the accumulator is still being computed
        for (int i = lane; i < wcols; i += 32) {
          const int col = c_first + (i >> 5) * c_step + (i & 31);
          const int n = n0 + col;
          const bool in = col < BN && n < p.N;
          wscale[i] = in ? p.s_x * __half2float(p.scale[n]) : 0.0f;
          wbias[i] = (in && p.bias != nullptr) ? __half2float(p.bias[n]) : 0.0f;
        }
      }
      if (!mbar_wait(&bar->acc_full[buf], (lt >> 1) & 1u, abort_flag, p.wait_ns)) {
        if (!*abort_flag) record_failure(bar, kDevErrTimeoutAccum);
        break;
      }
      tc_fence_after();
      __syncwarp();
      const uint32_t tacc = t_row + static_cast<uint32_t>(buf * p.acc_stride);
      // the 32-column chunks that hold valid output columns (a ragged last N tile has fewer)
      const int ncols = min(BN, tile_mma_n(p, tc));
      int kc = 0;   // chunk index of this warp within the tile
      if (c_first >= ncols) {
        // no chunk of this tile for this warp: the accumulator buffer is free at once
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar->acc_empty[buf]);
      }
      for (int c0 = c_first; c0 < ncols; c0 += c_step, ++chunk, ++kc) {
        const float* csc = wscale + kc * 32;
        const float* cbi = wbias + kc * 32;
        uint32_t r[32];
        tmem_ld_32x32b_x32(tacc + static_cast<uint32_t>(c0), r);
        tmem_wait_ld();
        if (c0 + c_step >= ncols) {
          // last read of this accumulator buffer: hand it back to the MMA warp
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bar->acc_empty[buf]);
        }
        if (p.cluster) {
          // this split's fp32 partial, row m of a [128][BN] tile in this CTA's shared
          // memory (the ring is idle: one tile per CTA and its MMAs are complete);
          // 16-byte chunks XOR-swizzled by the row so a warp's stores spread over banks
          const int m = q * 32 + lane;
          uint8_t* prow = smem + m * (BN * 4) + c0 * 4;
#pragma unroll
          for (int j = 0; j < 8; ++j)
            *reinterpret_cast<float4*>(prow + ((j ^ (m & 7)) << 4)) =
                make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                            __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
          continue;
        }
        uint8_t* dst = wbuf + (nbuf == 2 ? (chunk & 1u) * epi_buf : 0u);
        if (lane == 0) {
          // the store that last read dst: two chunks ago (two buffers) or the previous one
          if (nbuf == 2)
            bulk_wait_group_read<1>();
          else
            bulk_wait_group_read<0>();
        }
        __syncwarp();
        if (f32) {
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float4 o;
            o.x = __uint_as_float(r[4 * j + 0]);
            o.y = __uint_as_float(r[4 * j + 1]);
            o.z = __uint_as_float(r[4 * j + 2]);
            o.w = __uint_as_float(r[4 * j + 3]);
            if (!raw) {
              const float4 sc = *reinterpret_cast<const float4*>(csc + 4 * j);
              const float4 bi = *reinterpret_cast<const float4*>(cbi + 4 * j);
              o.x = fmaf(o.x, sc.x, bi.x);
              o.y = fmaf(o.y, sc.y, bi.y);
              o.z = fmaf(o.z, sc.z, bi.z);
              o.w = fmaf(o.w, sc.w, bi.w);
            }
            *reinterpret_cast<float4*>(dst + lane * 128 + ((j ^ (lane & 7)) << 4)) = o;
          }
        } else if (p.out_q8) {
          // fp16 value of the output (as a separate quantizer would read it), then
          // the 8-bit activation rule with the next layer's scale: 32 bytes per row.
          // The fast path covers all but values near a rounding tie (rare): those
          // are redone with the exact quotient.
          // 16 values at a time on the fast path (straight-line code the compiler can
          // interleave); a value near a tie (exact ties are common when s has few
          // significant bits) is redone alone with the exact quotient.
          uint32_t wq[8];
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            __half2 h[8];
            uint32_t qb[16];
            bool fast = true;
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
              const int j = 4 * hf + jj;
              const float4 sc = *reinterpret_cast<const float4*>(csc + 4 * j);
              const float4 bi = *reinterpret_cast<const float4*>(cbi + 4 * j);
              h[2 * jj] = __floats2half2_rn(fmaf(__uint_as_float(r[4 * j + 0]), sc.x, bi.x),
                                            fmaf(__uint_as_float(r[4 * j + 1]), sc.y, bi.y));
              h[2 * jj + 1] = __floats2half2_rn(fmaf(__uint_as_float(r[4 * j + 2]), sc.z, bi.z),
                                                fmaf(__uint_as_float(r[4 * j + 3]), sc.w, bi.w));
              const float2 x01 = __half22float2(h[2 * jj]);
              const float2 x23 = __half22float2(h[2 * jj + 1]);
              fast &= quant_fast_bits(x01.x, rs_out, qb[4 * jj + 0]);
              fast &= quant_fast_bits(x01.y, rs_out, qb[4 * jj + 1]);
              fast &= quant_fast_bits(x23.x, rs_out, qb[4 * jj + 2]);
              fast &= quant_fast_bits(x23.y, rs_out, qb[4 * jj + 3]);
            }
            if (!fast) quant_fix16(h, qb, p.s_out, rs_out);
#pragma unroll
            for (int jj = 0; jj < 4; ++jj)
              wq[4 * hf + jj] = pack_low_bytes(qb[4 * jj], qb[4 * jj + 1], qb[4 * jj + 2], qb[4 * jj + 3]);
          }
          if (p.out_q8 == kOutCodesF16) {
            // the codes as fp16 values (exact), staged like the fp16 output: 16-byte piece j
            // holds columns 8j .. 8j+7
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint32_t f0, f1, f2, f3;
              i8x4_to_f16x4(wq[2 * j], f0, f1);
              i8x4_to_f16x4(wq[2 * j + 1], f2, f3);
              *reinterpret_cast<uint4*>(dst + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) =
                  make_uint4(f0, f1, f2, f3);
            }
          } else {
            uint4* row = reinterpret_cast<uint4*>(dst + lane * 32);
            row[0] = make_uint4(wq[0], wq[1], wq[2], wq[3]);
            row[1] = make_uint4(wq[4], wq[5], wq[6], wq[7]);
          }
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float4 sc0 = *reinterpret_cast<const float4*>(csc + 8 * j);
            const float4 sc1 = *reinterpret_cast<const float4*>(csc + 8 * j + 4);
            const float4 bi0 = *reinterpret_cast<const float4*>(cbi + 8 * j);
            const float4 bi1 = *reinterpret_cast<const float4*>(cbi + 8 * j + 4);
            const float* rr = reinterpret_cast<const float*>(r) + 8 * j;
            __half2 h0 = __floats2half2_rn(fmaf(rr[0], sc0.x, bi0.x), fmaf(rr[1], sc0.y, bi0.y));
            __half2 h1 = __floats2half2_rn(fmaf(rr[2], sc0.z, bi0.z), fmaf(rr[3], sc0.w, bi0.w));
            __half2 h2 = __floats2half2_rn(fmaf(rr[4], sc1.x, bi1.x), fmaf(rr[5], sc1.y, bi1.y));
            __half2 h3 = __floats2half2_rn(fmaf(rr[6], sc1.z, bi1.z), fmaf(rr[7], sc1.w, bi1.w));
            *reinterpret_cast<uint4*>(dst + lane * 64 + ((j ^ ((lane >> 1) & 3)) << 4)) =
                make_uint4(*reinterpret_cast<uint32_t*>(&h0), *reinterpret_cast<uint32_t*>(&h1),
                           *reinterpret_cast<uint32_t*>(&h2), *reinterpret_cast<uint32_t*>(&h3));
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (raw)
            tma_store_3d(&mapY, dst, n0 + c0, m0 + q * 32, tc.split);
          else
            tma_store_2d(&mapY, dst, n0 + c0, m0 + q * 32);
          bulk_commit_group();
        }
        __syncwarp();
      }
    }
    if (lane == 0) bulk_wait_group_all();
  } else if (!kA16 && p.fused) {
    // ================================================================ decoders (fused path)
    // Each decoded group (8 consecutive k of one output row) is written as one
    // 16-byte chunk of the 128B-swizzled K-major B stage, so W-hat never leaves
    // shared memory.  Same arithmetic as the decode kernel: fp32 sum of the M
    // codewords in ascending m, one round to fp16.
    const int dt = threadIdx.x - 320;
    const int copy = lane & (fused_book_copies(p.M) - 1);   // this lane's codebook copy
    if (p.book_bytes > 0) {
      // 8-bit codebooks live in shared memory for the whole kernel, R copies of each
      // entry (staged by the decoders alone, while the producer's first loads are in
      // flight); thread i writes copy (r + i) % R at step r, so the stores of a quarter
      // warp land in distinct bank groups
      const int R = fused_book_copies(p.M);
      const uint4* gb = reinterpret_cast<const uint4*>(p.books);
      for (int i = dt; i < p.M * 256; i += kDecodeThreads) {
        const uint4 v = gb[i];
        for (int r = 0; r < R; ++r) sbook[i * R + ((r + i) & (R - 1))] = v;
      }
      named_barrier_sync(1, kDecodeThreads);
    }
    const int eb = p.B >> 3;                         // bytes per code
    const int G = p.K >> 3;
    Ring rg;
    bool failed = false;
    for (int t = blockIdx.x; t < p.total_tiles && !failed; t += gridDim.x) {
      const TileCoord tc = tile_coord(p, t);
      const int n0 = tc.n_tile * BN;
      for (int kb = tc.kb_begin; kb < tc.kb_end; kb += kStageBlocks) {
        const int nb = min(kStageBlocks, tc.kb_end - kb);
        // the producer copies a stage's codes only after the stage is free, so their
        // arrival also means the B stage may be overwritten
        if (!mbar_wait(&bar->codes_full[rg.s], rg.ph, abort_flag, p.wait_ns)) {
          if (!*abort_flag) record_failure(bar, kDevErrTimeoutFull);
          failed = true;
          break;
        }
        uint8_t* b_dst = bring + rg.s * b_stage;
        const uint8_t* c_src = scodes + rg.s * code_stage;
        // unit = (64-wide K block h, output row n): its 8 groups' codes are contiguous
        // (8*M*eb bytes, 8-byte aligned) and are read with vector loads.
        const int units = nb * BN;
        for (int u = dt; u < units; u += kDecodeThreads) {
          const int h = u / BN;
          const int n = u - h * BN;
          const int grow = n0 + n;
          const int gk0 = (kb + h) * 8;                // first group of this K block
          uint8_t* rowp = b_dst + h * b_half + n * 128;
          if (grow >= p.N || gk0 >= G) {
#pragma unroll
            for (int j = 0; j < 8; ++j)
              *reinterpret_cast<uint4*>(rowp + ((j ^ (n & 7)) << 4)) = make_uint4(0u, 0u, 0u, 0u);
            continue;
          }
          const uint8_t* cp = c_src + u * code_bytes;
          decode_unit_dispatch(p.M, eb, cp, sbook, reinterpret_cast<const uint4*>(p.books), rowp,
                               n, min(8, G - gk0), copy);
        }
        fence_proxy_async_smem();     // generic writes -> visible to the tensor core
        __syncwarp();
        if (lane == 0) mbar_arrive(&bar->full[rg.s]);
        rg.next(S);
      }
    }
  }

  if (p.cluster) {
    // In-cluster split-K reduction: CTA rank r of the cluster owns rows [r*rows, (r+1)*rows)
    // of the tile and sums them over the splits' shared-memory partials in split order
    // (the order of the split-K reduce kernel, so both give the same bits), then applies
    // the epilogue.  Every thread of every CTA passes both cluster barriers, also after a
    // failed wait above, so no CTA waits on a peer that left.
    __syncwarp();
    const TileCoord tc = tile_coord(p, blockIdx.x);
    const int nsp = p.splits;
    const int rows = (kBM + nsp - 1) / nsp;
    const int r0 = tc.split * rows;
    const int r1 = min(kBM, r0 + rows);
    const int c4n = BN >> 2;
    const int m0 = tc.m_tile * kBM;
    const int n0 = tc.n_tile * BN;
    const uint32_t pbase = smem_u32(smem);
    const int items = r1 > r0 ? (r1 - r0) * c4n : 0;
    cluster_sync_all();  // every split's partial tile is in its CTA's shared memory
    for (int i = threadIdx.x; i < items; i += blockDim.x) {
      const int mr = i / c4n;
      const int c4 = i - mr * c4n;
      const int m = r0 + mr;
      const int t = m0 + m;
      const int n = n0 + 4 * c4;
      if (t >= p.T || n >= p.N) continue;
      const uint32_t off =
          static_cast<uint32_t>(m * (BN * 4) + (c4 >> 3) * 128 + (((c4 & 7) ^ (m & 7)) << 4));
      float4 v[kMaxClusterSplits];
#pragma unroll
      for (int sp = 0; sp < kMaxClusterSplits; ++sp)
        if (sp < nsp) v[sp] = ld_cluster_f4(cluster_map(pbase + off, static_cast<uint32_t>(sp)));
      // the outputs' scale and bias are read while the partials are in flight
      float sc[4], bi[4];
      load_scale_bias4(p, n, sc, bi);
      float4 acc = v[0];
#pragma unroll
      for (int sp = 1; sp < kMaxClusterSplits; ++sp) {
        if (sp < nsp) {
          acc.x += v[sp].x;
          acc.y += v[sp].y;
          acc.z += v[sp].z;
          acc.w += v[sp].w;
        }
      }
      store_out4_sb(p, t, n, acc, sc, bi);
    }
    __syncwarp();
    cluster_sync_all();  // no CTA leaves while a peer still reads its shared memory
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
  grid_dependency_wait();
  allow_dependents();
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < nq;
       q += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = q / (p.N / 4);
    const int n = static_cast<int>(q - t * (p.N / 4)) * 4;
    float4 acc = *reinterpret_cast<const float4*>(p.partial + t * p.N + n);
    for (int s = 1; s < splits; ++s) {
      const float4 v = *reinterpret_cast<const float4*>(
          p.partial + (static_cast<int64_t>(s) * p.T + t) * p.N + n);
      acc.x += v.x;
      acc.y += v.y;
      acc.z += v.z;
      acc.w += v.w;
    }
    store_out4(p, t, static_cast<int>(n), acc);
  }
}

// Sum of many partials over few outputs (the table path: up to hundreds of chunks, one to four
// tokens): a block takes 32 output quads; warp j sums splits j, j + 8, j + 16, ... in order
// (independent loads in flight), then warp 0 adds the eight warps' sums in order and applies
// the epilogue.  The order is fixed, so results are reproducible.
__global__ void __launch_bounds__(256) lut_reduce_kernel(const GemmParams p, int splits) {
  // 16 output quads x 16 split groups per block: group j sums splits j, j + 16, ... with up to
  // four loads in flight, then group 0 adds the 16 group sums in order
  __shared__ float4 part[16][16];
  grid_dependency_wait();
  allow_dependents();
  const int qi = threadIdx.x & 15;
  const int j = threadIdx.x >> 4;
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  for (int64_t q0 = static_cast<int64_t>(blockIdx.x) * 16; q0 < nq;
       q0 += static_cast<int64_t>(gridDim.x) * 16) {
    const int64_t q = q0 + qi;
    const int64_t t = q / (p.N / 4);
    const int n = static_cast<int>(q - t * (p.N / 4)) * 4;
    float4 acc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    if (q < nq) {
      const float* base = p.partial + t * p.N + n;
      const int64_t stride = static_cast<int64_t>(p.T) * p.N;
      int s = j;
      for (; s + 48 < splits; s += 64) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          v[u] = *reinterpret_cast<const float4*>(base + (s + 16 * u) * stride);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc.x += v[u].x;
          acc.y += v[u].y;
          acc.z += v[u].z;
          acc.w += v[u].w;
        }
      }
      for (; s < splits; s += 16) {
        const float4 v = *reinterpret_cast<const float4*>(base + s * stride);
        acc.x += v.x;
        acc.y += v.y;
        acc.z += v.z;
        acc.w += v.w;
      }
    }
    part[j][qi] = acc;
    __syncthreads();
    if (j == 0 && q < nq) {
      float4 sum = part[0][qi];
#pragma unroll
      for (int w = 1; w < 16; ++w) {
        const float4 v = part[w][qi];
        sum.x += v.x;
        sum.y += v.y;
        sum.z += v.z;
        sum.w += v.w;
      }
      store_out4(p, t, n, sum);
    }
    __syncthreads();
  }
}

cudaError_t launch_lut_reduce(const GemmParams& p, int splits, cudaStream_t st) {
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  int64_t blocks = (nq + 15) / 16;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  return launch_pdl(lut_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, p,
                    splits);
}

cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, const CUtensorMap& mapY,
                        const GemmParams& p, int grid, cudaStream_t st) {
  static std::atomic<int> configured_i8[64] = {};
  static std::atomic<int> configured_a16[64] = {};
  const bool a16 = p.a16 != 0;
  // the shared-memory A form: dense weights only, 1 or 2 K blocks per stage, and the
  // TMEM holds just the two accumulators; the TMEM-A form needs two A slots beside them
  if (a16 && (p.fused || (p.sb != 1 && p.sb != 2) || 2 * p.BN > kTmemCols))
    return cudaErrorInvalidConfiguration;
  if (!a16 && (p.BN > kA8MaxBN || 2 * p.acc_stride + 2 * kASlotCols > kTmemCols))
    return cudaErrorInvalidConfiguration;
  if (p.BN % 32 != 0 || p.BN < 32 || p.BN > kMaxBN || p.stages < 1 || p.stages > kMaxStages)
    return cudaErrorInvalidConfiguration;
  const size_t bytes =
      gemm_smem_bytes(p.BN, p.stages, p.out_f32 || p.partial != nullptr, p.book_bytes,
                      p.fused ? 8 * p.M * (p.B >> 3) : 0, p.epi_warps, a16, p.sb);
  auto kernel = a16 ? aq_gemm_kernel<true> : aq_gemm_kernel<false>;
  const cudaError_t se = ensure_dynamic_smem(kernel, bytes, a16 ? configured_a16 : configured_i8);
  if (se != cudaSuccess) return se;
  // the decoder warps (10..15) exist only on the fused path; 12 epilogue warps only in the
  // shared-memory A form (2 + 12 warps within the kernel's thread bound)
  if (p.epi_warps != 4 && !(p.epi_warps == 8 && !p.fused && p.BN >= 64) &&
      !(p.epi_warps == 12 && a16 && p.BN >= 64))
    return cudaErrorInvalidConfiguration;
  // fp16 A form: producer, MMA and epilogue warps
  const int threads = a16 ? 32 * (2 + p.epi_warps) : (p.fused ? kThreads : 32 * (6 + p.epi_warps));
  if (!p.cluster)
    return launch_pdl(kernel, dim3(grid), dim3(threads), bytes, st, mapA, mapB, mapY, p);
  // in-cluster split-K: one CTA per (tile, split), the splits of a tile in one cluster
  if (p.splits < 2 || p.splits > kMaxClusterSplits || grid != p.total_tiles ||
      grid % p.splits != 0)
    return cudaErrorInvalidConfiguration;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = bytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(p.splits);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, mapA, mapB, mapY, p);
}

cudaError_t launch_splitk_reduce(const GemmParams& p, int splits, cudaStream_t st) {
  const int64_t nq = static_cast<int64_t>(p.T) * (p.N / 4);
  int64_t blocks = (nq + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  return launch_pdl(splitk_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, p,
                    splits);
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
