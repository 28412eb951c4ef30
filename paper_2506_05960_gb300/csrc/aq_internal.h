// aq_internal.h -- host-side declarations shared by the library's translation units.
#pragma once

#include <atomic>
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <utility>

namespace aq {

// ---- tile geometry of the tensor-core GEMM
constexpr int kBM = 128;        // rows (tokens / output pixels) per tile = TMEM lanes
constexpr int kBK = 64;         // K per TMA box / swizzle row (128 bytes of fp16)
constexpr int kStageBlocks = 2; // 64-wide K blocks per pipeline stage (8 MMAs of K = 16)
constexpr int kMaxBN = 256;     // widest N tile: 2 fp32 accumulators in TMEM
constexpr int kA8MaxBN = 192;   // the TMEM-A form also needs >= 2 A slots beside them
// GemmParams::out_q8 / SkinnyParams::out_q8: 0 (fp16 or fp32 output), or the 8-bit activation
// rule applied to the fp16-rounded output and stored as int8 codes or as their fp16 values
constexpr int kOutCodesI8 = 1;
constexpr int kOutCodesF16 = 2;
constexpr int kMaxStages = 8;   // pipeline ring depth bound
constexpr int kMaxClusterSplits = 8;  // K splits summed inside one cluster (portable size)

// Fused path, 8-bit codes: copies of the codebooks kept in shared memory.  A 16-byte
// load is served one quarter warp (8 lanes) per shared-memory cycle, and random codes
// make those lanes collide on banks.  Copy r stores entry e in 16-byte slot e * R + r
// and lane l reads copy l % R, so with R = 8 the 8 lanes of a quarter warp always hit
// 8 different bank groups.  Fewer copies for more codebooks keep the table <= 64 KB.
__host__ __device__ constexpr int fused_book_copies(int M) {
  return M <= 2 ? 8 : (M <= 4 ? 4 : 2);
}

// Parameters of one GEMM launch (passed by value).
struct GemmParams {
  int T, N, K;                  // rows, output channels, reduction length
  int BN;                       // N tile (multiple of 32, <= kMaxBN)
  int a16;                      // 1: A is fp16 in global memory (the 8-bit codes as fp16
                                // integers), TMA-loaded with the 128-byte swizzle and read by
                                // the MMA from shared memory; no converter warps.  0: int8 A,
                                // converted into a TMEM A ring
  int sb;                       // 64-wide K blocks per pipeline stage (a16: 1 or 2; else 2)
  int num_kb;                   // ceil(K / 64)
  int kb_per_split;             // K blocks per split
  int m_tiles, n_tiles, splits, total_tiles;
  int stages;                   // smem ring depth (TMA stages of 128 K)
  int a_stages;                 // TMEM A ring depth (slots of 128 K = 64 columns)
  int acc_stride, a_col;        // TMEM columns: accumulator buffer stride, first A slot
  // implicit-GEMM convolution (conv != 0): A is loaded per tap with a 4-D TMA box
  int conv, cin_blocks, pad, stride, tiles_per_img, rows_per_tile, imgs_per_tile;
  // epilogue
  float s_x;
  const __half* scale;
  const __half* bias;           // may be null
  void* y;
  int out_f32;
  int out_q8;                   // the next layer's activations, quantized with s_out: int8
                                // codes (kOutCodesI8) or the codes as fp16 values (kOutCodesF16)
  float s_out;
  float* partial;               // split-K partial sums [splits][T][N] (null: fused epilogue)
  int epi_warps;                // epilogue warps: 4, or 8 on the dense path (BN >= 64)
  int cluster;                  // 1: the splits of a tile form one thread-block cluster (split =
                                // cluster rank) and are summed through distributed shared
                                // memory; grid = total_tiles, one tile per CTA
  // fused decode (B stages written by decoder warps instead of TMA from a decoded W)
  int fused;
  const void* codes;            // packed codes
  const void* books;            // codebooks [M][2^B][8] fp16
  int M, B;
  int book_bytes;               // codebooks staged in shared memory (8-bit codes), else 0
  unsigned long long wait_ns;   // a pipeline wait gives up after this long (the error word
                                // then records which; drains always wait the full ~2 s)
};

// Parameters of the lookup-table kernel (linear layer, 8-bit codes, T <= 16).
constexpr int kLutrMaxCtas = 160;  // grid limit of the rotated-table kernel (one CTA per SM)

struct LutParams {
  const int8_t* xq;             // [T][K]
  const uint8_t* packed;        // packed codes [K/64][N][8][M]
  const __half* books;          // [M][256][8]
  float* partial;               // [chunks][T][N] partial sums
  int T, K, N, M;
  int vec;                      // 2: lutr_kernel (rotated, bank-conflict-free tables; Tp = 1,
                                // 2 or 4; M = 1, 2 or 4); 1: lutv_kernel (one token, any M,
                                // whole K blocks per chunk); 0: lut_kernel
  int Tp;                       // floats per table entry: vec: 1, 2 or 4 (>= T); else T
                                // rounded up to 4, 8 or 16
  int J;                        // groups per chunk (vec: whole K blocks; else divides 8)
  int G;                        // K / 8
  int chunks, rows_per_cta;
  int ctas;                     // lutr_kernel: grid size (at most kLutrMaxCtas)
  unsigned lutr_table_off;      // lutr_kernel: dynamic shared-memory offset of the tables (set
                                // by launch_lut so that they start at a 64 KB boundary)
  // lutr_kernel: CTA b takes the (chunk, 32-row block) units [unit_bounds[b], unit_bounds[b+1])
  // of the chunk-major order (contiguous ranges, balanced by the host for lookups plus builds)
  int64_t unit_bounds[kLutrMaxCtas + 1];
};

// Parameters of the few-token kernel (linear layer, T <= 16, one pass, no workspace).
struct SkinnyParams {
  const int8_t* xq;             // [T][K]
  const void* codes;            // packed codes [K/64][N][8][M]
  const void* books;            // [M][2^B][8] fp16
  const __half* scale;
  const __half* bias;           // may be null
  void* y;                      // [T][N]
  int out_f32, out_q8;          // out_q8: as GemmParams::out_q8
  float s_x, s_out;
  int T, K, N, M, B;
  int sms;                      // SMs of the device (the caller's count; sizes the grid)
  int x_smem;                   // set by the launcher: activations staged in shared memory
};

// Launch with programmatic stream serialization (the kernel must call
// grid_dependency_wait() before touching global memory).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// cudaFuncSetAttribute(MaxDynamicSharedMemorySize) applies to the current device: the
// size set so far is kept per device (0..63; others are set on every call) and raised
// only when a launch needs more.
template <typename Kernel>
cudaError_t ensure_dynamic_smem(Kernel kernel, size_t bytes, std::atomic<int> (&configured)[64]) {
  if (bytes <= 48 * 1024) return cudaSuccess;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const bool tracked = dev >= 0 && dev < 64;
  if (tracked && configured[dev].load() >= static_cast<int>(bytes)) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(bytes));
  if (e == cudaSuccess && tracked) {
    int cur = configured[dev].load();
    while (cur < static_cast<int>(bytes) &&
           !configured[dev].compare_exchange_weak(cur, static_cast<int>(bytes))) {
    }
  }
  return e;
}

// Launchers (return the launch status; they never synchronise).
cudaError_t launch_quant_act(const void* x, int8_t* xq, int64_t numel, float s, cudaStream_t st);
// The same rule, each 8-bit code stored as the fp16 value of that integer (exact).
cudaError_t launch_quant_act_f16(const void* x, __half* xh, int64_t numel, float s,
                                 cudaStream_t st);
cudaError_t launch_pack(const void* canon, void* packed, int N, int K, int M, int B,
                        cudaStream_t st);
cudaError_t launch_decode(const void* packed, const void* books, void* W, int N, int K, int M,
                          int B, cudaStream_t st);
// Wt[k][n] = fp16(scale[n] * W-hat[n][k]) (transposed, scaled decode for the input
// gradient) and ones[0..K) = 1 (the gradient GEMM's unit epilogue scale).
cudaError_t launch_decode_t(const void* packed, const void* books, const __half* scale,
                            __half* Wt, __half* ones, int N, int K, int M, int B,
                            cudaStream_t st);
// dC[m][c][e] += sum over groups with code c of s_x*scale[n]*G[n][group element e]
cudaError_t launch_codebook_grad(const void* codes, const float* G, const __half* scale,
                                 float s_x, float* dC, int N, int K, int g, int M, int B,
                                 cudaStream_t st);
// One greedy code-search step over codebooks [m_first, m_first + m_count) (8-bit
// codes, g = 8, canonical codes [N][K/8][M] updated in place).
cudaError_t launch_code_update(const float* W, const void* books, void* codes, const float* H,
                               int m_first, int m_count, int N, int K, int M, cudaStream_t st);
// Kernel-aware grouping (g = 9, 3x3 conv): codes [N][Cin][M], books [M][2^B][9] ->
// W [N][9*Cin] in the convolution's OHWI K order.
cudaError_t launch_decode_kaq(const void* codes, const void* books, void* W, int N, int Cin, int M,
                              int B, cudaStream_t st);
// code_bytes: packed code bytes per row and 64-wide K block staged per stage on
// the fused path (8 * M * bytes per code), 0 on the dense path.
// a16, sb: the shared-memory A form and its K blocks per stage (GemmParams).
size_t gemm_smem_bytes(int BN, int stages, bool f32_out, int book_bytes, int code_bytes,
                       int epi_warps, bool a16 = false, int sb = 2);
int gemm_max_stages(int BN, bool f32_out, int book_bytes, int code_bytes,
                    int epi_warps, bool a16 = false, int sb = 2);   // ring depth that fits
int gemm_a_stages(int BN);                   // TMEM A slots beside two BN-column accumulators
cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, const CUtensorMap& mapY,
                        const GemmParams& p, int grid, cudaStream_t st);
cudaError_t launch_splitk_reduce(const GemmParams& p, int splits, cudaStream_t st);
// The table path's chunk partials [splits][T][N]: summed by split groups in parallel (a fixed
// order), then the epilogue of launch_splitk_reduce.
cudaError_t launch_lut_reduce(const GemmParams& p, int splits, cudaStream_t st);
cudaError_t launch_lut(const LutParams& p, cudaStream_t st);
cudaError_t launch_skinny(SkinnyParams p, cudaStream_t st);

// Device error words of each translation unit (read and cleared, synchronising).
cudaError_t read_clear_gemm_error(unsigned* out);
cudaError_t read_clear_lut_error(unsigned* out);

}  // namespace aq
