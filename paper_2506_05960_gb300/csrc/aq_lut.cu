// aq_lut.cu -- lookup-table order of the AQ x A8 layer for small token counts
// (App. A.1, Eq. A5 -> A6, restated for a linear layer):
//   L[t][i][m][c] = sum_{e<g} x[t][g*i + e] * C^(m)[c][e]     for every codeword c
//   acc[t][n]     = sum_i sum_m L[t][i][m][ b[n][i][m] ]
// The weight matrix is never decoded: each output row costs M table reads per
// group instead of g multiply-adds, and the tables cost 2*g*M*2^B flops per
// group and token.  Only 8-bit codes (256-row codebooks) are supported.
// Three kernels, all writing fp32 partial sums per chunk of groups to the
// workspace [chunks][T][N] (a reduction applies scale and bias):
//   lutr_kernel  up to four tokens, M = 1, 2 or 4: bank-conflict-free rotated
//                tables, codes streamed per lane with cp.async (the AUTO choice);
//   lutv_kernel  one token, any other M;
//   lut_kernel   up to sixteen tokens, any M (on request).
//
// lut_kernel: one CTA owns a chunk of J consecutive groups (inside one packed
// 64-wide K block) and a slice of output rows: it stages the chunk's int8
// activations, builds the chunk's tables for all tokens in shared memory, then
// each thread walks its rows, reads the rows' codes with one contiguous load and
// gather-sums the table entries of all tokens (Tp floats per entry, 16-byte
// shared loads).
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

// One token with any number of codebooks (the rotated-table kernel below takes M = 1, 2 or 4):
// the same order with chunks of whole packed K blocks (two for M <= 4, else one) and one thread
// per output row, which reads its codes per K block as M contiguous 8-byte pieces (consecutive
// rows consecutive, so a warp's loads are coalesced) and adds one table entry per code, in the
// fixed order (K block, group, codebook).
__global__ void __launch_bounds__(256) lutv_kernel(const LutParams p) {
  extern __shared__ float4 lut_smem4[];
  float* L = reinterpret_cast<float*>(lut_smem4);              // [J][M][256]
  const int J = p.J, M = p.M;
  float* xs = L + static_cast<size_t>(J) * M * 256;            // [J * 8]
  grid_dependency_wait();
  allow_dependents();
  const int chunk = blockIdx.x;
  const int g0 = chunk * J;
  const int nj = min(J, p.G - g0);
  for (int e = threadIdx.x; e < J * 8; e += blockDim.x)
    xs[e] = e < nj * 8 ? static_cast<float>(p.xq[g0 * 8 + e]) : 0.0f;
  __syncthreads();
  // build: L[j][m][c] = sum_e x[g0 + j][e] * C^(m)[c][e], ascending e (zero past the last group)
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
    const float* xr = xs + j * 8;
    float s = 0.0f;
#pragma unroll
    for (int e = 0; e < 8; ++e) s = fmaf(xr[e], cw[e], s);
    L[ent] = s;
  }
  __syncthreads();
  const int kb0 = g0 >> 3;
  const int nkb = (nj + 7) >> 3;                  // packed K blocks holding this chunk's groups
  const int n_begin = blockIdx.y * p.rows_per_cta;
  const int n_end = min(p.N, n_begin + p.rows_per_cta);
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
          // byte pc*8 + k of the record is group (pc*8 + k) / M, codebook (pc*8 + k) % M
          const uint32_t code = ((k < 4 ? v.x : v.y) >> (8 * (k & 3))) & 0xFFu;
          acc += Lb[(pc * 8 + k) * 256 + code];
        }
      }
    }
    p.partial[static_cast<int64_t>(chunk) * p.N + n] = acc;
  }
}

// ------------------------------------------------------------------------------------------
// Rotated-table kernel: one to four tokens, M = 1, 2 or 4 codebooks of 2^8 entries.  The table
// order of App. A.1 (Eq. A5 -> A6) with tables laid out so that the lanes of a warp never
// collide on a shared-memory bank, whatever the codes:
//  * a chunk is NT = 32 / TP consecutive bytes of every row's code stream (the row's packed
//    records of consecutive K blocks, 8 * M bytes each: stream byte b is group b / M, codebook
//    b % M), i.e. NT tables, one per (group, codebook);
//  * entry e of table t (TP floats, one per token) is stored at word e * 64 + t * TP and again
//    at word e * 64 + (t + NT) * TP: 256 rows of 64 words, 64 KB, placed at shared-window
//    address kLutrTableAddr (a multiple of 64 KB);
//  * lane l owns one output row; at step s (0 <= s < NT) it adds the entry of table
//    (l' + s) mod NT, l' = l mod NT, read from slot l' + s < 2 NT (the copy spares the wrap).
//    The lanes of one shared-memory phase (32 / TP lanes, distinct l') read TP-word slots
//    (l' + s) * TP mod 32 that are pairwise distinct: one conflict-free wavefront per phase;
//  * the row's NT code bytes are rotated by l' bytes once (whole 8-byte steps by the order in
//    which the ring's 8-byte slots are read, then one word select and a funnel shift), so step
//    s takes byte s of the rotated words, and one byte permute assembles the entry's whole
//    shared address: kLutrTableAddr | code << 8 | l' * TP * 4 (plus s * TP * 4 as the load's
//    offset).
// Each lane sums its row's entries in its own rotated order (fixed per lane: deterministic).
// Work: (chunk, 32-row block) units in chunk-major order, one contiguous range per CTA (one CTA
// per SM), the ranges set by the host so that the busiest CTA's lookups plus table builds are as
// few as it can make them: a CTA builds the tables of each chunk its range reaches from
// codebooks staged once in shared memory (widened to fp32 there when they fit), and writes fp32
// partial sums [chunk][T][N]; the reduction sums the chunks and applies the epilogue.
// Start-up: before the grid-dependency wait, one thread asks L2 to prefetch the codebooks and
// the codes of every warp's first kStages row blocks; after it, one cp.async group brings the
// codebooks and the activations of the first two chunks, ahead of the code stream's groups.
// Code streaming: every lane copies its own row's NT code bytes with cp.async into a private
// ring of kLutrLaneRing bytes (kStages row blocks ahead, across chunk boundaries) and reads them
// back after waiting for its own copies: each lane touches only what it copied, so no barrier
// is needed, and a warp keeps several row blocks of codes in flight.
constexpr int kLutrThreads = 1024;
constexpr int kLutrLaneRing = 96;                // bytes of code ring per lane
constexpr uint32_t kLutrTableAddr = 0x20000u;    // shared-window address of the tables

__device__ unsigned g_lut_err = 0;               // AQ_DEVERR_* bits of the table kernels

template <int MM, int TP>
struct LutrShape {
  static constexpr int NT = 32 / TP;             // tables (code bytes of a row) per chunk
  static constexpr int NW = NT / 4;              // 32-bit code words of a row per chunk
  static constexpr int R = 8 * MM;               // bytes of one packed record (row, K block)
  static constexpr int GC = NT / MM;             // groups per chunk
  static constexpr int PB = NT < R ? NT : R;
  static constexpr int P = PB < 16 ? PB : 16;    // bytes per code copy
  static constexpr int NP = NT / P;              // copies per row and chunk
  static constexpr int kStages = kLutrLaneRing / NT;
  static constexpr uint32_t kRingBytes = static_cast<uint32_t>(kLutrThreads) * kLutrLaneRing;
  static constexpr uint32_t kStageBytes = static_cast<uint32_t>(kLutrThreads) * NT;
  static constexpr uint32_t kBookOff = kRingBytes;
  // the codebooks widened to fp32 once per CTA (when they fit before the tables)
  static constexpr bool kBookF32 = MM <= 2;
  static constexpr uint32_t kBookFOff = kBookOff + MM * 256 * 16;
  static constexpr uint32_t kXsOff = kBookFOff + (kBookF32 ? MM * 256 * 32 : 0);
  static constexpr int kXq = TP * GC * 8;        // activation bytes of one chunk
  static constexpr uint32_t kXq8Off = kXsOff + (kXq * 4 + 15) / 16 * 16;
  static constexpr uint32_t kFront = kXq8Off + 2 * ((kXq + 15) / 16 * 16);
  static constexpr uint32_t kTableBytes = 256 * 64 * 4;
};

__device__ __forceinline__ void cp_async_zfill(uint32_t dst, const void* src, bool valid,
                                               int bytes) {
  const int n = valid ? bytes : 0;               // 0: nothing is read, the bytes are zeroed
  if (bytes == 16)
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
                 : "memory");
  else
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(n)
                 : "memory");
}

template <int MM, int TP>
__global__ void __launch_bounds__(kLutrThreads, 1) lutr_kernel(const LutParams p) {
  using S = LutrShape<MM, TP>;
  constexpr int NT = S::NT, NW = S::NW, R = S::R, GC = S::GC, P = S::P, NP = S::NP;
  constexpr int D = S::kStages;
  extern __shared__ float4 lut_smem4[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(lut_smem4);
  const uint32_t sbase = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  // the host sized the allocation for this base; any other layout would misplace the tables
  if (sbase + p.lutr_table_off != kLutrTableAddr || p.lutr_table_off < S::kFront) {
    if (threadIdx.x == 0) atomicOr(&g_lut_err, kDevErrSmemLayout);
    return;
  }
  uint4* sbook = reinterpret_cast<uint4*>(smem + S::kBookOff);                  // [MM][256]
  float* xs = reinterpret_cast<float*>(smem + S::kXsOff);                       // [TP][GC*8]
  float* L = reinterpret_cast<float*>(smem + p.lutr_table_off);                 // [256][64]
  const int N = p.N, T = p.T;
  const int KB = (p.K + 63) / 64;
  const int64_t stream_bytes = static_cast<int64_t>(KB) * R;   // code bytes of a row
  const int nrb = (N + 31) / 32;
  const int64_t u0 = p.unit_bounds[blockIdx.x];
  const int64_t u1 = p.unit_bounds[blockIdx.x + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nwarps = blockDim.x >> 5;
  const int c_first = static_cast<int>(u0 / nrb);
  const int rb_first = static_cast<int>(u0 % nrb);
  const int c_last = static_cast<int>((u1 - 1) / nrb);
  const int rb_last_end = static_cast<int>((u1 - 1) % nrb) + 1;
  if (u0 < u1 && threadIdx.x == 0) {
    // the codebooks and the first kStages row blocks of every warp (contiguous rows of the
    // first chunk) start moving into L2 while the previous kernel still runs: a prefetch only
    // warms the cache and every read of the data comes after the wait below, so this holds
    // even if that kernel wrote them
    bulk_prefetch_l2(p.books, MM * 256 * 16);
    const int64_t total16 = (static_cast<int64_t>(KB) * N * R) & ~static_cast<int64_t>(15);
    const int rb_stop = c_first == c_last ? rb_last_end : nrb;
    const int rb_end = rb_first + nwarps * D < rb_stop ? rb_first + nwarps * D : rb_stop;
    const int64_t r0 = static_cast<int64_t>(rb_first) * 32;
    const int64_t r_end = static_cast<int64_t>(rb_end) * 32;
    const int64_t r1 = r_end < N ? r_end : N;
    const int64_t b0 = static_cast<int64_t>(c_first) * NT;
    const int64_t b1 = b0 + NT < stream_bytes ? b0 + NT : stream_bytes;
    for (int64_t pl = b0 / R; pl * R < b1; ++pl) {
      // these rows' whole records of the plane, widened to 16-byte bounds inside the buffer
      const int64_t a0 = ((pl * N + r0) * R) & ~static_cast<int64_t>(15);
      int64_t a1 = ((pl * N + r1) * R + 15) & ~static_cast<int64_t>(15);
      if (a1 > total16) a1 = total16;
      if (a1 > a0) bulk_prefetch_l2(p.packed + a0, static_cast<uint32_t>(a1 - a0));
    }
  }
  grid_dependency_wait();
  allow_dependents();
  if (u0 >= u1) return;
  const int li = lane & (NT - 1);
  // entry address = kLutrTableAddr | code << 8 | lane_off (bytes 2, 0 of lane_reg; byte 1 from
  // the code)
  const uint32_t lane_reg = kLutrTableAddr | static_cast<uint32_t>(li * TP * 4);

  // ---- producer: this warp's row blocks, chunk by chunk (rb_begin(c) + warp, + nwarps, ...),
  // copied kStages items ahead of the lookups; every lane of the warp walks the same sequence
  int pc = c_first, prb = rb_first + warp;       // next item to copy
  const uint8_t* psrc = p.packed;                // its piece-0 source for this lane's row
  uint32_t pmask = 0;                            // its pieces inside the code stream
  auto prod_settle = [&]() {
    while (pc <= c_last && prb >= (pc == c_last ? rb_last_end : nrb)) {
      ++pc;
      prb = warp;
    }
    if (pc <= c_last) {
      const int64_t b0 = static_cast<int64_t>(pc) * NT;
      psrc = p.packed + ((b0 / R) * N + prb * 32 + lane) * R + (b0 % R);
      pmask = 0;
#pragma unroll
      for (int q = 0; q < NP; ++q)
        if (b0 + q * P < stream_bytes) pmask |= 1u << q;
    }
  };
  prod_settle();
  const uint32_t ring_lane = sbase + static_cast<uint32_t>(threadIdx.x * P);
  // the row's chunk as NS 8-byte slots: slot i of the registers is read from ring slot
  // (i + li / 8) mod NS, which is the rotation by whole 8-byte slots
  constexpr int NS = NT / 8;
  uint32_t slot_addr[NS];
#pragma unroll
  for (int i = 0; i < NS; ++i) {
    const int j = (i + (li >> 3)) & (NS - 1);
    slot_addr[i] =
        ring_lane + static_cast<uint32_t>((j * 8 / P) * kLutrThreads * P + (j * 8) % P);
  }
  uint32_t wr = 0;                               // write offset of the next stage
  auto produce = [&]() {
    if (pc <= c_last) {
      const bool row_ok = prb * 32 + lane < N;
#pragma unroll
      for (int q = 0; q < NP; ++q) {
        const bool ok = row_ok && ((pmask >> q) & 1u);
        // piece q: q * P bytes further in the stream: the next record, or further in this one
        const int64_t poff = static_cast<int64_t>((q * P) / R) * N * R + (q * P) % R;
        cp_async_zfill(ring_lane + wr + static_cast<uint32_t>(q * kLutrThreads * P),
                       ok ? psrc + poff : p.packed, ok, P);
      }
      prb += nwarps;
      if (prb < (pc == c_last ? rb_last_end : nrb))
        psrc += static_cast<int64_t>(nwarps) * 32 * R;
      else
        prod_settle();
    }
    asm volatile("cp.async.commit_group;" ::: "memory");   // empty past the end: counts stay
    wr += S::kStageBytes;
    if (wr == S::kRingBytes) wr = 0;
  };
  // the codebooks and the first chunk's activations: one copy group ahead of the code stream
  {
    const uint32_t sb = sbase + S::kBookOff;
    for (int i = threadIdx.x; i < MM * 256; i += blockDim.x)
      cp_async_zfill(sb + i * 16, reinterpret_cast<const uint4*>(p.books) + i, true, 16);
    constexpr int kPieces = S::kXq / 16;           // per chunk; the first two chunks
    if (threadIdx.x < 2 * kPieces) {
      const int h = threadIdx.x / kPieces;
      const int i = threadIdx.x - h * kPieces;
      const int tt = i / (GC * 8 / 16);
      const int k = (c_first + h) * GC * 8 + (i % (GC * 8 / 16)) * 16;
      const bool ok = tt < T && k < p.K;         // K % 16 == 0: a piece is all in or all out
      cp_async_zfill(sbase + S::kXq8Off + threadIdx.x * 16,
                     ok ? p.xq + static_cast<int64_t>(tt) * p.K + k : p.xq, ok, 16);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  }
#pragma unroll 1
  for (int d = 0; d < D; ++d) produce();
  uint32_t rd = 0;                               // read offset of the oldest stage
  asm volatile("cp.async.wait_group %0;" ::"n"(D) : "memory");
  __syncthreads();
  float4* sbookf = reinterpret_cast<float4*>(smem + S::kBookFOff);          // [MM][256][2]
  if constexpr (S::kBookF32) {
    for (int i = threadIdx.x; i < MM * 256; i += blockDim.x) {
      const uint4 raw = sbook[i];
      const __half2* h2 = reinterpret_cast<const __half2*>(&raw);
      const float2 f0 = __half22float2(h2[0]), f1 = __half22float2(h2[1]);
      const float2 f2 = __half22float2(h2[2]), f3 = __half22float2(h2[3]);
      sbookf[2 * i] = make_float4(f0.x, f0.y, f1.x, f1.y);
      sbookf[2 * i + 1] = make_float4(f2.x, f2.y, f3.x, f3.y);
    }
  }

  for (int c = c_first; c <= c_last; ++c) {
    const int g0 = c * GC;                       // first group of the chunk
    // ---- the chunk's tables (after every warp is done with the previous chunk's)
    __syncthreads();
    if (c <= c_first + 1) {
      const int8_t* xq8 = reinterpret_cast<const int8_t*>(smem + S::kXq8Off) + (c - c_first) * S::kXq;
      for (int i = threadIdx.x; i < TP * GC * 8; i += blockDim.x) xs[i] = static_cast<float>(xq8[i]);
    } else {
      for (int i = threadIdx.x; i < TP * GC * 8; i += blockDim.x) {
        const int tt = i / (GC * 8);
        const int k = g0 * 8 + (i - tt * GC * 8);
        xs[i] = (tt < T && k < p.K) ? static_cast<float>(p.xq[static_cast<int64_t>(tt) * p.K + k])
                                    : 0.0f;
      }
    }
    __syncthreads();
    {
      const int t = threadIdx.x % NT;
      const int j = t / MM;                      // group within the chunk
      const bool live = g0 + j < p.G;            // groups past K (zero-padded codes): 0
      float xr[TP][8];
#pragma unroll
      for (int tt = 0; tt < TP; ++tt)
#pragma unroll
        for (int e = 0; e < 8; ++e) xr[tt][e] = xs[tt * GC * 8 + j * 8 + e];
      const uint4* book = sbook + (t % MM) * 256;
#pragma unroll 2
      for (int e = threadIdx.x / NT; e < 256; e += kLutrThreads / NT) {
        float o[TP];
#pragma unroll
        for (int tt = 0; tt < TP; ++tt) o[tt] = 0.0f;
        if (live) {
          // L[e] = sum_u x[g0 + j][u] * C^(m)[e][u], ascending u (the other table kernels'
          // arithmetic)
          float cw[8];
          if constexpr (S::kBookF32) {
            const float4 a = sbookf[((t % MM) * 256 + e) * 2];
            const float4 b = sbookf[((t % MM) * 256 + e) * 2 + 1];
            cw[0] = a.x; cw[1] = a.y; cw[2] = a.z; cw[3] = a.w;
            cw[4] = b.x; cw[5] = b.y; cw[6] = b.z; cw[7] = b.w;
          } else {
            const uint4 raw = book[e];
            const __half2* h2 = reinterpret_cast<const __half2*>(&raw);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float2 f = __half22float2(h2[i]);
              cw[2 * i] = f.x;
              cw[2 * i + 1] = f.y;
            }
          }
#pragma unroll
          for (int tt = 0; tt < TP; ++tt) {
            float s = 0.0f;
#pragma unroll
            for (int v = 0; v < 8; ++v) s = fmaf(xr[tt][v], cw[v], s);
            o[tt] = s;
          }
        }
        float* d0 = L + e * 64 + t * TP;
        float* d1 = d0 + NT * TP;
        if constexpr (TP == 1) {
          d0[0] = o[0];
          d1[0] = o[0];
        } else if constexpr (TP == 2) {
          *reinterpret_cast<float2*>(d0) = make_float2(o[0], o[1]);
          *reinterpret_cast<float2*>(d1) = make_float2(o[0], o[1]);
        } else {
          *reinterpret_cast<float4*>(d0) = make_float4(o[0], o[1], o[2], o[3]);
          *reinterpret_cast<float4*>(d1) = make_float4(o[0], o[1], o[2], o[3]);
        }
      }
    }
    __syncthreads();
    const int rb_e = c == c_last ? rb_last_end : nrb;
    float* pout = p.partial + static_cast<int64_t>(c) * T * N + lane;
    for (int rb = (c == c_first ? rb_first : 0) + warp; rb < rb_e; rb += nwarps) {
      // this row block's codes: the oldest of this lane's copy groups
      asm volatile("cp.async.wait_group %0;" ::"n"(D - 1) : "memory");
      uint32_t r[NW];
#pragma unroll
      for (int i = 0; i < NS; ++i)
        asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];"
                     : "=r"(r[2 * i]), "=r"(r[2 * i + 1]) : "r"(slot_addr[i] + rd) : "memory");
      // rotate the row's code bytes left by li: byte s of r is stream byte (s + li) mod NT (the
      // slots above rotated by whole 8 bytes; one word step and a funnel shift remain)
      if ((li >> 2) & 1) {
        uint32_t tmp[NW];
#pragma unroll
        for (int k = 0; k < NW; ++k) tmp[k] = r[(k + 1) % NW];
#pragma unroll
        for (int k = 0; k < NW; ++k) r[k] = tmp[k];
      }
      {
        const uint32_t sh = static_cast<uint32_t>(8 * (li & 3));
        uint32_t tmp[NW];
#pragma unroll
        for (int k = 0; k < NW; ++k) tmp[k] = __funnelshift_r(r[k], r[(k + 1) % NW], sh);
#pragma unroll
        for (int k = 0; k < NW; ++k) r[k] = tmp[k];
      }
      // the stage is free again (its words are in registers and used above): refill it with
      // this warp's item kStages ahead
      produce();
      rd += S::kStageBytes;
      if (rd == S::kRingBytes) rd = 0;
      // two running sums (even and odd steps), each started by its first entry
      float acc0[TP], acc1[TP];
#pragma unroll
      for (int s = 0; s < NT; ++s) {
        const uint32_t addr = __byte_perm(r[s >> 2], lane_reg, 0x7604u | ((s & 3) << 4)) +
                              static_cast<uint32_t>(s * TP * 4);
        float* acc = (s & 1) ? acc1 : acc0;
        float v[TP];
        if constexpr (TP == 1) {
          asm("ld.shared.f32 %0, [%1];" : "=f"(v[0]) : "r"(addr));
        } else if constexpr (TP == 2) {
          asm("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v[0]), "=f"(v[1]) : "r"(addr));
        } else {
          asm("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
              : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]) : "r"(addr));
        }
#pragma unroll
        for (int tt = 0; tt < TP; ++tt) acc[tt] = s < 2 ? v[tt] : acc[tt] + v[tt];
      }
      if (rb * 32 + lane < N) {
#pragma unroll
        for (int tt = 0; tt < TP; ++tt)
          if (tt < T) pout[static_cast<int64_t>(tt) * N + rb * 32] = acc0[tt] + acc1[tt];
      }
    }
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// Dynamic shared memory of lutr_kernel for a window whose dynamic part starts at `base`: the
// ring, codebooks and activations, then the tables at kLutrTableAddr.  0 if they do not fit.
static uint32_t lutr_front(int TP, int M) {
  switch (TP * 16 + M) {
    case 16 + 1: return LutrShape<1, 1>::kFront;
    case 16 + 2: return LutrShape<2, 1>::kFront;
    case 16 + 4: return LutrShape<4, 1>::kFront;
    case 32 + 1: return LutrShape<1, 2>::kFront;
    case 32 + 2: return LutrShape<2, 2>::kFront;
    case 32 + 4: return LutrShape<4, 2>::kFront;
    case 64 + 1: return LutrShape<1, 4>::kFront;
    case 64 + 2: return LutrShape<2, 4>::kFront;
    case 64 + 4: return LutrShape<4, 4>::kFront;
    default: return 0;
  }
}

size_t lut_smem_bytes(int J, int M, int Tp, int T) {
  return static_cast<size_t>(J) * M * 256 * Tp * 4 + static_cast<size_t>(T) * J * 8 * 4;
}

cudaError_t read_clear_lut_error(unsigned* out) {
  unsigned v = 0;
  cudaError_t e = cudaMemcpyFromSymbol(&v, g_lut_err, sizeof(v));
  if (e != cudaSuccess) return e;
  const unsigned zero = 0;
  e = cudaMemcpyToSymbol(g_lut_err, &zero, sizeof(zero));
  *out = v;
  return e;
}

cudaError_t launch_lut(const LutParams& p, cudaStream_t st) {
  if (p.vec == 2) {
    // lutr_kernel: p.Tp floats per entry, p.ctas CTAs of 1024 threads
    static std::atomic<int> c11[64] = {}, c21[64] = {}, c41[64] = {}, c12[64] = {}, c22[64] = {},
                            c42[64] = {}, c14[64] = {}, c24[64] = {}, c44[64] = {};
    // the dynamic window starts after the per-block reserved shared memory (no static shared
    // memory in this kernel): the tables go at kLutrTableAddr, the rest before them
    int dev = 0, reserved = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess)
      e = cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
    if (e != cudaSuccess) return e;
    const uint32_t front = lutr_front(p.Tp, p.M);
    if (front == 0 || static_cast<uint32_t>(reserved) + front > kLutrTableAddr)
      return cudaErrorInvalidConfiguration;
    LutParams q = p;
    q.lutr_table_off = kLutrTableAddr - static_cast<uint32_t>(reserved);
    const size_t bytes = q.lutr_table_off + 256 * 64 * 4;
    auto go = [&](auto kernel, std::atomic<int> (&conf)[64]) -> cudaError_t {
      const cudaError_t se = ensure_dynamic_smem(kernel, bytes, conf);
      if (se != cudaSuccess) return se;
      return launch_pdl(kernel, dim3(static_cast<unsigned>(q.ctas)), dim3(1024), bytes, st, q);
    };
    switch (p.Tp * 16 + p.M) {
      case 16 + 1: return go(lutr_kernel<1, 1>, c11);
      case 16 + 2: return go(lutr_kernel<2, 1>, c21);
      case 16 + 4: return go(lutr_kernel<4, 1>, c41);
      case 32 + 1: return go(lutr_kernel<1, 2>, c12);
      case 32 + 2: return go(lutr_kernel<2, 2>, c22);
      case 32 + 4: return go(lutr_kernel<4, 2>, c42);
      case 64 + 1: return go(lutr_kernel<1, 4>, c14);
      case 64 + 2: return go(lutr_kernel<2, 4>, c24);
      case 64 + 4: return go(lutr_kernel<4, 4>, c44);
      default: return cudaErrorInvalidConfiguration;
    }
  }
  if (p.vec == 1) {
    // lutv_kernel: one token, whole K blocks per chunk
    static std::atomic<int> conf[64] = {};
    const size_t bytes = static_cast<size_t>(p.J) * p.M * 256 * 4 + static_cast<size_t>(p.J) * 8 * 4;
    const int n_slices = (p.N + p.rows_per_cta - 1) / p.rows_per_cta;
    const cudaError_t se = ensure_dynamic_smem(lutv_kernel, bytes, conf);
    if (se != cudaSuccess) return se;
    return launch_pdl(lutv_kernel, dim3(p.chunks, n_slices), dim3(256), bytes, st, p);
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
