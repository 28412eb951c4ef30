// aq_internal.h -- host-side declarations shared by the library's translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

namespace aq {

// ---- tile geometry of the tensor-core GEMM
constexpr int kBM = 128;        // rows (tokens / output pixels) per tile = TMEM lanes
constexpr int kBK = 64;         // K per pipeline stage (128 bytes of fp16 = one swizzle row)
constexpr int kMaxBN = 256;     // widest N tile (TMEM columns of the fp32 accumulator)

// Parameters of one GEMM launch (passed by value).
struct GemmParams {
  int T, N, K;                  // rows, output channels, reduction length
  int BN;                       // N tile (multiple of 16, <= 256)
  int num_kb;                   // ceil(K / 64)
  int kb_per_split;             // K blocks per split (grid.z splits)
  // implicit-GEMM convolution (conv != 0): A is loaded per tap with a 4-D TMA box
  int conv, cin_blocks, pad, tiles_per_img, rows_per_tile, imgs_per_tile;
  // epilogue
  float s_x;
  const __half* scale;
  const __half* bias;           // may be null
  void* y;
  int out_f32;
  float* partial;               // split-K partial sums [splits][T][N] (null: fused epilogue)
};

// Launchers (return the launch status; they never synchronise).
cudaError_t launch_quant_act(const void* x, int8_t* xq, int64_t numel, float s, cudaStream_t st);
cudaError_t launch_pack(const void* canon, void* packed, int N, int K, int M, int B,
                        cudaStream_t st);
cudaError_t launch_decode(const void* packed, const void* books, void* W, int N, int K, int M,
                          int B, cudaStream_t st);
cudaError_t launch_gemm(const CUtensorMap& mapA, const CUtensorMap& mapB, const GemmParams& p,
                        int n_tiles, int m_tiles, int splits, cudaStream_t st);
cudaError_t launch_splitk_reduce(const GemmParams& p, int splits, cudaStream_t st);

// Device error words of each translation unit (read and cleared, synchronising).
cudaError_t read_clear_gemm_error(unsigned* out);

}  // namespace aq
