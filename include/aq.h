/*
 * aq.h -- C ABI of the GB300 (sm_103a) additive-quantized (AQ) weight x
 * 8-bit activation (A8) layer library.
 *
 * The method (AQUATIC-Diff, arXiv 2506.05960) stores every linear and
 * convolution weight of a diffusion UNet in the additive-quantization format
 * of Sec. 2.4, Eq. 4: the weight matrix is cut row-major into groups of g
 * consecutive weights, and each group is the sum of M codewords, one from each
 * codebook C^(m) (2^B rows of g entries), selected by the M codes b[i, m] of
 * the group.  Activations are quantized to 8 bits with one scale per call
 * (one per denoising timestep, Sec. 4.2.3).  A convolution is the same
 * contraction over the im2col matrix (Sec. 3.1.1), computed here as an
 * implicit GEMM without materialising im2col.
 *
 * Conventions shared by every entry point
 *   - All array pointers are DEVICE pointers owned by the caller.  The library
 *     allocates no device memory and never synchronises the device; each call
 *     only enqueues kernels on `stream` (a cudaStream_t, NULL = legacy default
 *     stream).  Inputs are not modified.
 *   - Sizes are element counts.  Arrays are dense, row-major, C-contiguous.
 *   - Every pointer must be 16-byte aligned (AQ_ERR_ALIGN otherwise).
 *   - Supported formats: g = 8; B = 8 with M in 1..8, or B = 16 with M in 1..2.
 *     g = 9 selects the kernel-aware grouping of a 3x3 convolution (Sec. 3.1.2,
 *     App. A.1 Eq. A4: one group = the 9 taps of one (output channel, input
 *     channel) filter); it is accepted by aq_packed_size, aq_pack, aq_decode,
 *     aq_conv2d_workspace_size and aq_conv2d_nhwc (dense path) only.
 *     Codes of B = 8 are uint8, codes of B = 16 are uint16 (little endian).
 *     Codebooks are fp16 [M][2^B][g].  Per-output-channel scale and bias are
 *     fp16 [N] (bias may be NULL).  The activation scale s_x is fp32.
 *   - Return value: AQ_OK (0) or a negative AQ_ERR_* code.  On error nothing
 *     is enqueued, and aq_last_error_string() describes the failure (text is
 *     per host thread, valid until the next call on that thread).
 *   - Device-side waits are bounded: a pipeline stage that does not complete
 *     in about two seconds sets a device error word and the kernel returns;
 *     aq_device_error() reads (and clears) that word.
 */
#ifndef AQ_H_
#define AQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AQ_ABI_VERSION 1

#if defined(__GNUC__)
#define AQ_API __attribute__((visibility("default")))
#else
#define AQ_API
#endif

/* ---- status codes ------------------------------------------------------ */
#define AQ_OK                    0
#define AQ_ERR_NULL             -1  /* a required pointer is NULL                      */
#define AQ_ERR_SHAPE            -2  /* a size is negative/zero where it must not be, or
                                       not a multiple of what the format needs           */
#define AQ_ERR_UNSUPPORTED      -3  /* (g, M, B), conv geometry or path not supported   */
#define AQ_ERR_ALIGN            -4  /* a pointer is not 16-byte aligned                 */
#define AQ_ERR_WORKSPACE        -5  /* workspace NULL or smaller than required          */
#define AQ_ERR_CUDA             -6  /* a CUDA runtime/driver call or launch failed      */
#define AQ_ERR_DEVICE_TIMEOUT   -7  /* a kernel gave up on a bounded wait               */

/* ---- enums --------------------------------------------------------------- */
typedef enum aq_dtype {
  AQ_DTYPE_F16 = 0,   /* output fp16, round to nearest even */
  AQ_DTYPE_F32 = 1,   /* output fp32                        */
  AQ_DTYPE_I8 = 2,    /* int8 codes of the 8-bit activation rule: output of the _q8 and
                         _ex calls (quantized with s_out); input of the _ex calls */
  AQ_DTYPE_F16_CODES = 3  /* the same codes held as fp16 values (exact): output and input
                             of the _ex calls; the layout the shared-memory A form reads */
} aq_dtype;

typedef enum aq_path {
  AQ_PATH_AUTO  = 0,  /* library picks from (T, N, K, M, B): linear layers with T <= 4 take
                         AQ_PATH_LUT when B = 8, the codes fill at least 6 MB and (T == 1
                         or M is 1, 2 or 4), else AQ_PATH_FEW_TOKENS; one 128-row tile of
                         tokens AQ_PATH_FUSED; more AQ_PATH_DENSE (a convolution: FUSED for
                         one tile with g = 8, else DENSE)                                  */
  AQ_PATH_DENSE = 1,  /* decode W-hat once into the workspace (Sec. 4.4: decompress, then
                         the ordinary layer op), then a TMA-fed tcgen05 tensor-core GEMM   */
  AQ_PATH_FUSED = 2,  /* decode inside the GEMM into shared memory (codebooks in shared
                         memory, or in L2 for 2^16-entry books); W-hat never touches HBM  */
  AQ_PATH_LUT   = 3,  /* lookup-table order of App. A.1 (Eq. A5-A6): per token and group,
                         the dot product with every codeword, then a gather-sum by code
                         (up to four tokens with M = 1, 2 or 4: bank-conflict-free rotated
                         tables); linear layers with T <= 16 and B = 8; needs a workspace
                         for the per-chunk partial sums                                    */
  AQ_PATH_FEW_TOKENS = 4, /* linear layers with T <= 16: one kernel streams each row's codes
                         once, decodes in registers and dots with every token on CUDA
                         cores; no workspace                                              */
  AQ_PATH_PREDECODED = 5  /* the dense path without its decode: the workspace's first
                         N*K fp16 values already hold W-hat, written by aq_decode with the
                         same codes and codebooks (e.g. on another stream, ahead of the
                         layer, while the previous layer runs); same workspace size and
                         plan as AQ_PATH_DENSE, same results                              */
} aq_path;

/* ---- library information -------------------------------------------------- */

/* ABI version of the loaded library (AQ_ABI_VERSION). */
AQ_API int aq_abi_version(void);

/* Text of the last error on the calling host thread ("" if none). */
AQ_API const char* aq_last_error_string(void);

/* Reads and clears the device error words of the current device (kernels set them
 * when a bounded wait gives up, or when a kernel finds its launch inconsistent and
 * skips its work).  Synchronises the device.  *code_out = 0 if no kernel reported an
 * error, else an OR of AQ_DEVERR_* bits.  Returns AQ_OK or AQ_ERR_CUDA. */
AQ_API int aq_device_error(int* code_out);
#define AQ_DEVERR_TIMEOUT_FULL   1   /* a consumer waited too long for a loaded stage      */
#define AQ_DEVERR_TIMEOUT_EMPTY  2   /* the loader waited too long for a free stage        */
#define AQ_DEVERR_TIMEOUT_CONV   4   /* the MMA waited too long for converted activations  */
#define AQ_DEVERR_TIMEOUT_ACCUM  8   /* the MMA or epilogue waited too long for an
                                        accumulator buffer                                  */
#define AQ_DEVERR_TIMEOUT_DRAIN 16   /* after a time-out, in-flight copies did not drain   */
#define AQ_DEVERR_SMEM_LAYOUT   32   /* the rotated-table kernel found its shared memory at
                                        another window address than its launch assumed, and
                                        skipped its work (the call's output is undefined)   */

/* Failure-path testing: later tensor-core launches of this host thread give up a
 * pipeline wait after ns nanoseconds (checked every 256 polls) instead of about two
 * seconds; ns < 0 restores the default.  A kernel that gives up records the
 * AQ_DEVERR_* bit, stops its other warps, waits (up to the default limit) for its
 * own copies and MMAs in flight, frees its tensor memory and returns: the call's
 * output is then undefined, the context stays usable and aq_device_error() reports
 * the bits.  Not for production use.  Always AQ_OK.                             */
AQ_API int aq_set_wait_limit_ns(int64_t ns);

/* ---- kernel timing (diagnostics) -------------------------------------------
 * When enabled, every entry point records a CUDA event pair on the caller's
 * stream around each kernel it launches; aq_profile_read() waits for the
 * recorded events and returns, per kernel kind, the summed device time in
 * milliseconds and the number of launches since the last aq_profile_enable().
 * Kinds: 0 quantizer, 1 pack, 2 decode, 3 tensor-core GEMM, 4 split-K reduce,
 * 5 LUT build, 6 LUT gather, 7 fused-decode GEMM.  Uses host-side CUDA events
 * only (no device memory).  Calls captured into a CUDA graph record external
 * event nodes: replay the graph once, then read (a read reports the last
 * replay).  Event creation happens on first use: make one uncaptured call
 * with timing enabled before capturing.                                      */
#define AQ_PROFILE_KINDS 8
AQ_API int aq_profile_enable(int on);
AQ_API int aq_profile_read(double* ms_out, int64_t* launches_out, int n_kinds);

/* ---- code packing (Eq. 4 codes b[i, m]) -------------------------------------
 * Canonical code layout: [N][K/g][M] (uint8 for B = 8, uint16 for B = 16), the
 * groups of each output row in order along K, the M codes of a group
 * contiguous.  Packed layout (storage format of every other entry point):
 * [ceil(K/64)][N][64/g][M], i.e. for each 64-wide block of K the codes that one
 * output row needs are contiguous (16 bytes for M = 2, B = 8) and consecutive
 * rows follow each other, so a warp reads a block of rows with 128-bit loads.
 * Codes of a zero-padded K tail are 0.
 * g = 9 (kernel-aware grouping, K = 9*Cin): canonical codes are [Cout][Cin][M]
 * and the packed layout is that same array (aq_pack copies it).              */

/* Bytes of the packed buffer for an N x K layer. */
AQ_API int aq_packed_size(int N, int K, int g, int M, int B, size_t* bytes);

/* Canonical codes -> packed codes (device to device; run once per layer). */
AQ_API int aq_pack(const void* codes_canon, void* codes_packed,
            int N, int K, int g, int M, int B, void* stream);

/* ---- decode (Sec. 2.4 Eq. 4; Sec. 4.4 "decompress prior to the layer op") --
 * W_out[n][k] = fp16( sum_{m=0..M-1} fp32(C^(m)[b[n, k/g, m]][k mod g]) ), the
 * fp32 sum taken in ascending m and rounded once to fp16 (round to nearest
 * even, overflow to +-inf, subnormals kept).  Bit-exact against that rule.
 * The per-channel scale is NOT folded in.  W_out is fp16 [N][K].
 * g = 9 (kernel-aware grouping): codebooks fp16 [M][2^B][9]; the group of
 * (n, c) holds the 9 taps t = i*3 + j of that filter and is written in the
 * convolution's OHWI order, W_out[n][t*Cin + c] with Cin = K/9 (same rule).   */
AQ_API int aq_decode(const void* codes_packed, const void* codebooks, void* W_out,
              int N, int K, int g, int M, int B, void* stream);

/* ---- codebook gradient (backward of Eq. 4; Sec. 3.2.1 continuous step) -----
 * The decoded group is the sum of its M codewords, so the gradient of a loss L
 * with respect to codeword row c of codebook m collects every group that uses
 * it:  dC[m][c][e] += sum_{(n, i): b[n, i, m] = c}  s_x * scale[n] * G[n][i*g + e]
 * where G[n][k] = dL/dW[n][k] for the unscaled decoded weight, i.e.
 * sum_t dY[t][n] * xq[t][k] (a plain GEMM of the output gradient and the
 * layer's int8 input, run by the caller).  g = 9: G is in the convolution's OHWI
 * order (element e of the (n, c) filter at column e*Cin + c).
 *   codes_packed  as for aq_decode;  G fp32 [N][K];  scale fp16 [N] or NULL (1);
 *   dC fp32 [M][2^B][g], ACCUMULATED (clear it first for a plain gradient).
 * Summation order is not fixed (atomic adds): results match the exact sum to
 * fp32 accumulation error, not bit for bit.                                    */
AQ_API int aq_codebook_grad(const void* codes_packed, const float* G, const void* scale,
                            float s_x, float* dC, int N, int K, int g, int M, int B,
                            void* stream);

/* ---- input gradient (backward of the layer; Sec. 3.2.1 continuous step) ----
 * dX[t][k] = alpha * sum_n dY[t][n] * scale[n] * W[n][k], W the decoded AQ weight.
 * With alpha = 1 this is the gradient with respect to the dequantized activations
 * X = s_x * xq of the layer y = diag(scale) W X + bias; alpha = s_x gives it with
 * respect to the 8-bit codes xq (the straight-through quantizer).  Computed as the
 * same decode + tensor-core contraction as the forward layer: a transposed decode
 * writes Wt[k][n] = fp16(scale[n] * W[n][k]) (W by the decode rule above, the product
 * rounded once more to fp16) into the workspace, then the fp16-activation GEMM
 * contracts dY with it over n, accumulating in fp32.
 *   dY fp16 [T][N]; codes, codebooks, scale as for aq_linear; dX [T][K] fp16 or fp32.
 *   K % 16 == 0, N % 16 == 0 (AQ_ERR_SHAPE); T == 0 is a no-op; alpha finite.
 *   Workspace: aq_linear_input_grad_workspace_size() bytes.                       */
AQ_API int aq_linear_input_grad_workspace_size(int T, int K, int N, int g, int M, int B,
                                               size_t* bytes);
AQ_API int aq_linear_input_grad(const void* dy, float alpha, const void* codes_packed,
                                const void* codebooks, const void* scale, void* dx,
                                int out_dtype, int T, int K, int N, int g, int M, int B,
                                void* workspace, size_t workspace_bytes, void* stream);

/* ---- code search step (Stage-1 calibration, Sec. 3.1) ---------------------
 * One greedy step of the code optimisation (beam width 1): for every group and
 * each codebook m in [m_first, m_first + m_count), in that order, b[m] becomes
 * the codeword that minimises the group's error with the other codes fixed:
 *   r = w - sum_{m' != m} C^(m')[b[m']] (ascending m'),  d = C^(m)[c] - r,
 *   score(c) = d^T H_i d,  ties to the lowest c,
 * where H_i is group column i's g x g block of A A^T for calibration inputs A
 * (the block-diagonal part of ||W A - W-hat A||^2), or the identity when H is
 * NULL.  Computed in fp32, every product and sum rounded separately, sums in
 * ascending element order; the result is bit-exact against that rule.
 *   W fp32 [N][K] target weight;  codebooks fp16 [M][256][8];
 *   codes uint8 CANONICAL [N][K/8][M], read and updated in place;
 *   H fp32 [K/8][8][8] or NULL.  g = 8 and B = 8 only.                     */
AQ_API int aq_code_update(const float* W, const void* codebooks, void* codes, const float* H,
                          int m_first, int m_count, int N, int K, int g, int M, int B,
                          void* stream);

/* ---- 8-bit activation quantizer (Sec. 4.2.3; symmetric form of Eq. 3) ------
 * xq[i] = clip(round_half_even(x[i] / s_x), -127, 127), x fp16, division in
 * IEEE fp32, NaN -> 0.  s_x must be finite and > 0 (AQ_ERR_SHAPE otherwise).
 * numel == 0 is a no-op.                                                     */
AQ_API int aq_quant_act(const void* x, int8_t* xq, int64_t numel, float s_x, void* stream);

/* ---- AQ x A8 linear layer --------------------------------------------------
 * y[t][n] = (s_x * scale[n]) * sum_k xq[t][k] * W[n][k] + bias[n]
 * with W = the decoded AQ weight (fp16 under the decode rule above),
 * products accumulated in fp32, the scale/bias epilogue in fp32, y fp16 (round
 * to nearest even) or fp32.
 *   xq      int8 [T][K]
 *   y       [T][N] of out_dtype
 *   T >= 0 (T == 0 is a no-op), K % 16 == 0, N % 8 == 0, N, K > 0.
 *   workspace: device scratch of at least aq_linear_workspace_size() bytes
 *   (may be NULL when that size is 0); contents on entry are ignored.
 *   path: AQ_PATH_* (AUTO recommended).                                       */
AQ_API int aq_linear_workspace_size(int T, int K, int N, int g, int M, int B, int path,
                             size_t* bytes);
/* Diagnostics: restrict the tensor-core plan of later calls made by this host
 * thread (workspace-size queries included) to N tile BN (0 = any), K splits
 * (0 = any) and in-cluster split sum (1), split-K through the workspace (0) or
 * either (-1).  A call whose shapes admit no such plan runs the cost-model plan
 * (int8 activations take BN <= 192; fp16 activations, BN <= 256).
 * aq_set_plan_override(0, 0, -1) restores the default.  AQ_ERR_SHAPE for a BN
 * that is not a multiple of 32 in [0, 256] or other out-of-range values.      */
AQ_API int aq_set_plan_override(int BN, int splits, int cluster);

/* Plan that aq_linear (fp16 or int8 output) runs for these shapes, for
 * diagnostics: info[0] = resolved AQ_PATH_*; for the tensor-core paths info[1] =
 * N tile, info[2] = K splits, info[3] = 1 when the splits of a tile are summed
 * inside one thread-block cluster (no partials in the workspace, no reduce
 * kernel), info[4] = pipeline stages, info[5] = (tile, split) work items,
 * info[6] = 1 when the tensor cores read fp16 activations from shared memory
 * (aq_linear_f16 and aq_linear_a16 on the dense paths; 0: int8 activations
 * converted into tensor memory), info[7] = 64-wide K blocks per pipeline stage;
 * for AQ_PATH_LUT info[2] = chunks of the code stream (fp32 partial sums per
 * output) and info[5] = CTAs of the rotated-table kernel (0 when another table
 * kernel runs; the launch takes at most the device's SM count); 0 for the other
 * paths and fields.  Writes min(n_info, 8) entries (zero past 8).  No
 * device access.  aq_linear_f16_plan / aq_linear_a16_plan: the plans of those
 * entry points.                                                                */
AQ_API int aq_linear_plan(int T, int K, int N, int g, int M, int B, int path, int* info,
                          int n_info);
AQ_API int aq_linear_f16_plan(int T, int K, int N, int g, int M, int B, int path, int* info,
                              int n_info);
AQ_API int aq_linear_a16_plan(int T, int K, int N, int g, int M, int B, int path, int* info,
                              int n_info);
AQ_API int aq_linear(const int8_t* xq, float s_x, const void* codes_packed,
              const void* codebooks, const void* scale, const void* bias,
              void* y, int out_dtype, int T, int K, int N, int g, int M, int B,
              void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- layer with the next layer's activation quantizer fused in ------------
 * yq[t][n] = clip(round_half_even(fp32(y16[t][n]) / s_out), -127, 127), where
 * y16 is the fp16 output aq_linear would write: the 8-bit activations of the
 * next layer (Sec. 4.2.3), produced in the layer's epilogue instead of by a
 * separate aq_quant_act pass over an fp16 tensor.  Bit-exact against
 * aq_linear (fp16) followed by aq_quant_act with s_out on the same path.
 *   yq int8 [T][N]; s_out finite and > 0; N % 16 == 0 (AQ_ERR_SHAPE).
 *   Workspace: aq_linear_workspace_size() (the same plan as fp16 output).
 * Other arguments, layouts and errors as for aq_linear.                     */
AQ_API int aq_linear_q8(const int8_t* xq, float s_x, const void* codes_packed,
                        const void* codebooks, const void* scale, const void* bias,
                        int8_t* yq, float s_out, int T, int K, int N, int g, int M, int B,
                        void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- layer from fp16 activations -------------------------------------------
 * aq_quant_act(x, xq, T*K, s_x) followed by aq_linear(xq, s_x, ...) in one call
 * (Sec. 4.2.3 quantizer, then the layer of Sec. 3.1.1).  The quantized activations
 * are kept at the start of the workspace: on the dense paths as fp16 values (each
 * 8-bit code exactly; the tensor cores then read both operands from shared
 * memory), on the other paths as int8.  Same codes as aq_quant_act; the output
 * equals the two calls' bit for bit when both run the same plan (N tile and K
 * split, aq_set_plan_override), and is within the layer tolerance otherwise.
 *   x fp16 [T][K]; s_x finite and > 0 (AQ_ERR_SHAPE); out_dtype F16 or F32.
 *   Workspace: aq_linear_f16_workspace_size() bytes = 2*T*K rounded up to 1 KB
 *   plus the layer's workspace for this plan; with AQ_PATH_PREDECODED, W-hat is
 *   expected right after that activation region (byte offset 2*T*K rounded up to
 *   1 KB).                                                                       */
AQ_API int aq_linear_f16_workspace_size(int T, int K, int N, int g, int M, int B, int path,
                                        size_t* bytes);
AQ_API int aq_linear_f16(const void* x, float s_x, const void* codes_packed,
                         const void* codebooks, const void* scale, const void* bias, void* y,
                         int out_dtype, int T, int K, int N, int g, int M, int B,
                         void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- layer on 8-bit activations stored as fp16 values -----------------------
 * aq_linear with xh[t][k] = fp16(xq[t][k]) (the codes of Sec. 4.2.3 held as fp16
 * integers, e.g. as written into aq_linear_f16's workspace): the tensor cores read
 * both operands from shared memory.  Any fp16 values are accepted and multiplied as
 * they are.  Paths: AUTO (= DENSE), DENSE, PREDECODED; others AQ_ERR_UNSUPPORTED.
 *   xh fp16 [T][K]; other arguments, layouts and errors as for aq_linear.
 *   Workspace: aq_linear_a16_workspace_size() bytes.                            */
AQ_API int aq_linear_a16_workspace_size(int T, int K, int N, int g, int M, int B, int path,
                                        size_t* bytes);
AQ_API int aq_linear_a16(const void* xh, float s_x, const void* codes_packed,
                         const void* codebooks, const void* scale, const void* bias, void* y,
                         int out_dtype, int T, int K, int N, int g, int M, int B,
                         void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- linear layer without any device allocation --------------------------
 * The paper has no counterpart: this is a deployment convenience.  Some callers
 * cannot call cudaMalloc at all (code running under a fixed memory budget that
 * is reserved up front, a host allocator that must not be re-entered from a
 * callback, or an engine that forbids allocation once it is serving), so they
 * cannot provide the workspace that aq_linear needs for the decoded weights.
 * aq_linear_noalloc gives the same result as aq_linear on the dense path
 * without K splitting (AQ_PATH_DENSE with aq_set_plan_override(0, 1, 0)), bit for
 * bit, and within the layer tolerance of aq_linear's other plans.  It decodes the
 * weights into a fixed scratch array that the library holds in device memory:
 * AQ_NOALLOC_SCRATCH_BYTES (16 MiB) per GPU that loads the library, kept until
 * the process exits.
 *   - Limit: N * K * 2 <= AQ_NOALLOC_SCRATCH_BYTES (N * K <= 8,388,608
 *     weights); larger layers return AQ_ERR_WORKSPACE before any CUDA call.
 *   - The first call on each device, and the first after that device's context
 *     was re-created (e.g. by cudaDeviceReset), looks up the array's device
 *     address with that device current; make such a call before any stream
 *     capture.  No call allocates or synchronises.
 *   - Every call shares the one array and overwrites what it uses (nothing
 *     in it needs to start at zero).  Calls that can overlap on the GPU (on
 *     different streams without ordering) race on the array and give wrong
 *     results: order them on one stream or with events.
 *   - Never calls cudaMalloc, cudaFree or any allocating library routine.
 * Arguments, layouts and other errors as for aq_linear.                     */
#define AQ_NOALLOC_SCRATCH_BYTES (16u << 20)
AQ_API int aq_linear_noalloc(const int8_t* xq, float s_x, const void* codes_packed,
                             const void* codebooks, const void* scale, const void* bias,
                             void* y, int out_dtype, int T, int K, int N, int g, int M, int B,
                             void* stream);

/* ---- AQ x A8 3x3 convolution, NHWC, implicit GEMM (Sec. 3.1.1) -------------
 * y[b][ho][wo][n] = (s_x*scale[n]) * sum_{i,j,c} xq[b][ho*s+i-pad][wo*s+j-pad][c]
 *                   * W[n][(i*kw + j)*Cin + c] + bias[n],
 * out-of-image taps read as 0.  The weight is the decoded AQ matrix [Cout][K]
 * with K = kh*kw*Cin in OHWI order, groups of g = 8 along Cin inside one tap,
 * or g = 9: one group per (n, c) filter (codes [Cout][Cin][M], dense path;
 * AQ_PATH_FUSED and AQ_PATH_LUT return AQ_ERR_UNSUPPORTED, AUTO picks dense).
 *   xq int8 [Nb][H][W][Cin];  y [Nb][Ho][Wo][Cout] of out_dtype,
 *   Ho = (H + 2*pad - kh)/stride + 1, Wo likewise.
 *   Supported: kh = kw = 3, pad = 1, stride 1 or 2, Cin % 64 == 0,
 *   Cout % 8 == 0.  A 1x1 convolution is aq_linear over the NHWC rows.       */
AQ_API int aq_conv2d_workspace_size(int Nb, int H, int W, int Cin, int Cout, int kh, int kw,
                             int stride, int pad, int g, int M, int B, int path,
                             size_t* bytes);
/* Plan of aq_conv2d_nhwc for these shapes; info as for aq_linear_plan.          */
AQ_API int aq_conv2d_plan(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride,
                          int pad, int g, int M, int B, int path, int* info, int n_info);
AQ_API int aq_conv2d_nhwc(const int8_t* xq, float s_x, const void* codes_packed,
                   const void* codebooks, const void* scale, const void* bias,
                   void* y, int out_dtype, int Nb, int H, int W, int Cin, int Cout,
                   int kh, int kw, int stride, int pad, int g, int M, int B,
                   void* workspace, size_t workspace_bytes, int path, void* stream);

/* The convolution with the next layer's quantizer fused in (as aq_linear_q8):
 * yq int8 [Nb][Ho][Wo][Cout], Cout % 16 == 0; workspace as for
 * aq_conv2d_workspace_size().                                                */
AQ_API int aq_conv2d_nhwc_q8(const int8_t* xq, float s_x, const void* codes_packed,
                             const void* codebooks, const void* scale, const void* bias,
                             int8_t* yq, float s_out, int Nb, int H, int W, int Cin, int Cout,
                             int kh, int kw, int stride, int pad, int g, int M, int B,
                             void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- 3x3 convolution from fp16 activations ---------------------------------
 * aq_quant_act(x, xq, Nb*H*W*Cin, s_x) followed by aq_conv2d_nhwc(xq, s_x, ...)
 * in one call (Sec. 4.2.3 quantizer, then the convolution above).  As for
 * aq_linear_f16, the quantized activations stay at the start of the workspace:
 * on the dense paths as fp16 values (each 8-bit code exactly), which the tensor
 * cores read from shared memory through 4-D NHWC boxes with the 128-byte
 * swizzle; on the fused path as int8.  Same codes as aq_quant_act; the output
 * equals the two calls' bit for bit when both run the same plan (N tile and K
 * split, aq_set_plan_override), and is within the layer tolerance otherwise.
 *   x fp16 [Nb][H][W][Cin]; s_x finite and > 0 (AQ_ERR_SHAPE); out_dtype F16 or
 *   F32 (AQ_DTYPE_I8: AQ_ERR_UNSUPPORTED).  Shapes, codes and the other arrays
 *   as for aq_conv2d_nhwc.
 *   Workspace: aq_conv2d_f16_workspace_size() bytes = 2*Nb*H*W*Cin rounded up
 *   to 1 KB, then the layer's workspace for this plan (with AQ_PATH_PREDECODED,
 *   W-hat is expected right after the activation region).
 *   aq_conv2d_f16_plan: the plan these calls run; info as for aq_linear_plan.  */
AQ_API int aq_conv2d_f16_workspace_size(int Nb, int H, int W, int Cin, int Cout, int kh,
                                        int kw, int stride, int pad, int g, int M, int B,
                                        int path, size_t* bytes);
AQ_API int aq_conv2d_f16_plan(int Nb, int H, int W, int Cin, int Cout, int kh, int kw,
                              int stride, int pad, int g, int M, int B, int path, int* info,
                              int n_info);
AQ_API int aq_conv2d_nhwc_f16(const void* x, float s_x, const void* codes_packed,
                              const void* codebooks, const void* scale, const void* bias,
                              void* y, int out_dtype, int Nb, int H, int W, int Cin, int Cout,
                              int kh, int kw, int stride, int pad, int g, int M, int B,
                              void* workspace, size_t workspace_bytes, int path, void* stream);

/* ---- layer calls with the activation and output kinds as arguments ----------
 * The linear layer / 3x3 convolution above, with
 *   act_dtype  AQ_DTYPE_I8: act holds int8 codes (as aq_linear / aq_conv2d_nhwc), or
 *              AQ_DTYPE_F16_CODES: act holds the codes as fp16 values (as aq_linear_a16); the
 *              tensor cores then read them from shared memory, on a dense path (AUTO means
 *              AQ_PATH_DENSE; AQ_PATH_FUSED, _LUT, _FEW_TOKENS: AQ_ERR_UNSUPPORTED);
 *   out_dtype  AQ_DTYPE_F16 or AQ_DTYPE_F32 (s_out unused), or AQ_DTYPE_I8 /
 *              AQ_DTYPE_F16_CODES: the next layer's codes under the activation rule with
 *              scale s_out applied to the fp16-rounded output (as aq_linear_q8), stored as
 *              int8 (N % 16 == 0) or as their fp16 values.
 * A chain of layers can so hand each layer its activations in the form its own plan reads
 * (aq_linear_f16_plan / aq_conv2d_f16_plan report, in info[6], whether the shared-memory A
 * form is the faster one for a shape).  The codes as fp16 values and as int8 give the same
 * bits when both run the same plan (N tile and K split).  Shapes, paths, workspace and
 * errors otherwise as for the calls above; act_dtype other than the two: AQ_ERR_UNSUPPORTED. */
AQ_API int aq_linear_ex_workspace_size(int act_dtype, int T, int K, int N, int g, int M, int B,
                                       int path, size_t* bytes);
AQ_API int aq_linear_ex_plan(int act_dtype, int T, int K, int N, int g, int M, int B, int path,
                             int* info, int n_info);
AQ_API int aq_linear_ex(const void* act, int act_dtype, float s_x, const void* codes_packed,
                        const void* codebooks, const void* scale, const void* bias, void* y,
                        int out_dtype, float s_out, int T, int K, int N, int g, int M, int B,
                        void* workspace, size_t workspace_bytes, int path, void* stream);
AQ_API int aq_conv2d_ex_workspace_size(int act_dtype, int Nb, int H, int W, int Cin, int Cout,
                                       int kh, int kw, int stride, int pad, int g, int M, int B,
                                       int path, size_t* bytes);
AQ_API int aq_conv2d_ex_plan(int act_dtype, int Nb, int H, int W, int Cin, int Cout, int kh,
                             int kw, int stride, int pad, int g, int M, int B, int path,
                             int* info, int n_info);
AQ_API int aq_conv2d_nhwc_ex(const void* act, int act_dtype, float s_x,
                             const void* codes_packed, const void* codebooks, const void* scale,
                             const void* bias, void* y, int out_dtype, float s_out, int Nb, int H,
                             int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g,
                             int M, int B, void* workspace, size_t workspace_bytes, int path,
                             void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AQ_H_ */
