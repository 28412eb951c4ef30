// aq_api.cu -- the C ABI declared in include/aq.h: argument validation, path
// and tile planning, TMA descriptor encoding, and kernel launches.  Nothing
// here allocates device memory or synchronises (except aq_device_error).
#include <algorithm>
#include <atomic>
#include <vector>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include <cuda.h>
#include <cuda_runtime.h>

#include "aq.h"
#include "aq_internal.h"
#include "aq_ptx.cuh"

// The kernels' error bits are the ones aq_device_error() documents.
static_assert(aq::kDevErrTimeoutFull == AQ_DEVERR_TIMEOUT_FULL &&
              aq::kDevErrTimeoutEmpty == AQ_DEVERR_TIMEOUT_EMPTY &&
              aq::kDevErrTimeoutConv == AQ_DEVERR_TIMEOUT_CONV &&
              aq::kDevErrTimeoutAccum == AQ_DEVERR_TIMEOUT_ACCUM &&
              aq::kDevErrTimeoutDrain == AQ_DEVERR_TIMEOUT_DRAIN &&
              aq::kDevErrSmemLayout == AQ_DEVERR_SMEM_LAYOUT,
              "device error bits differ from aq.h");

// Scratch of aq_linear_noalloc: the decoded weights of one call.  Lives for the
// life of the process on every device that loads this module.
static __device__ __align__(256) unsigned char g_noalloc_scratch[AQ_NOALLOC_SCRATCH_BYTES];

namespace {

thread_local std::string g_last_error;

int set_error(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return code;
}

int ok() {
  g_last_error.clear();
  return AQ_OK;
}

int cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return ok();
  return set_error(AQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// ---- format checks (g, M, B).  g = 9 is the kernel-aware grouping of a 3x3 conv
// (one group per (output channel, input channel) filter); only the entry points
// that can take it pass allow_kaq.
constexpr int kKaqGroup = 9;

int check_format(int g, int M, int B, bool allow_kaq = false) {
  if (g != 8 && !(allow_kaq && g == kKaqGroup))
    return set_error(AQ_ERR_UNSUPPORTED,
                     allow_kaq ? "group size g=%d unsupported (8, or 9 for 3x3 convolutions)"
                               : "group size g=%d unsupported here (g=8)",
                     g);
  if (B == 8) {
    if (M < 1 || M > 8) return set_error(AQ_ERR_UNSUPPORTED, "M=%d unsupported for B=8 (1..8)", M);
  } else if (B == 16) {
    if (M < 1 || M > 2) return set_error(AQ_ERR_UNSUPPORTED, "M=%d unsupported for B=16 (1..2)", M);
  } else {
    return set_error(AQ_ERR_UNSUPPORTED, "B=%d unsupported (8 or 16)", B);
  }
  return AQ_OK;
}

// ---- cuTensorMapEncodeTiled through the runtime's driver entry point
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = []() -> EncodeTiledFn {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    return reinterpret_cast<EncodeTiledFn>(p);
  }();
  return fn;
}

// elem_strides (optional): traversal stride per dimension; a box dimension of
// size b with traversal stride s delivers b / s elements (b a multiple of s).
int encode(CUtensorMap* map, CUtensorMapDataType dt, int rank, const void* base,
           const cuuint64_t* dims, const cuuint64_t* strides, const cuuint32_t* box,
           CUtensorMapSwizzle sw, const cuuint32_t* elem_strides = nullptr) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return set_error(AQ_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  cuuint32_t es[5] = {1, 1, 1, 1, 1};
  if (elem_strides)
    for (int i = 0; i < rank; ++i) es[i] = elem_strides[i];
  CUresult r = fn(map, dt, static_cast<cuuint32_t>(rank), const_cast<void*>(base), dims, strides,
                  box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_error(AQ_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return AQ_OK;
}

// ---- GEMM planning (no device queries: the plan, and so the workspace size,
// depends only on the shapes)
constexpr int kPlanSMs = 152;            // GB300 SM count assumed by the cost model
constexpr size_t kSmemOptin = 232448;    // max dynamic shared memory per CTA on sm_103

// Clusters of S CTAs (one CTA per SM) resident at once, S = 0..8, as reported by
// cudaOccupancyMaxActiveClusters on GB300 (152 SMs): the GPC layout leaves fewer
// than 152 / S.  A plan whose clusters exceed this runs in two waves.
constexpr int kPlanMaxClusters[aq::kMaxClusterSplits + 1] = {0, 152, 76, 46, 36, 28, 23, 15, 15};

struct Plan {
  int BN, n_tiles, m_tiles, splits, kb_per_split, num_kb;
  int stages, a_stages, acc_stride, a_col, total_tiles;
  int cluster;    // the splits of a tile form one cluster and are summed in shared memory
  int epi_warps;  // 4, or 8 on the dense path with fp16/int8 staging and BN >= 64
  int a16;        // A is fp16 in global memory (the 8-bit codes as fp16 values)
  int sb;         // 64-wide K blocks per pipeline stage
};

// K blocks per stage of the shared-memory A form (a stage is then one fp16 A box and
// one weight box: more, shallower stages than the TMEM-A form's 128-wide ones).
#ifndef AQ_A16_STAGE_BLOCKS
#define AQ_A16_STAGE_BLOCKS 1
#endif
constexpr int kA16StageBlocks = AQ_A16_STAGE_BLOCKS;

// Cycles of one pipeline stage (eight 128 x BN x 16 MMAs issued by one thread),
// measured on GB300: an MMA takes BN/2 cycles (at least 48; N = 160 runs at 88),
// and the stage's barrier wait + commits hide under the MMAs only from BN = 192.
double stage_cycles(int BN) {
  double mma = BN == 160 ? 88.0 : (BN / 2.0 < 48.0 ? 48.0 : BN / 2.0);
  double exposed = BN >= 192 ? 0.0 : (BN >= 160 ? 60.0 : 115.0);
  return 8.0 * mma + exposed;
}

// The fp16 A form, per 128 of K (two 64-wide K blocks, each one pipeline stage of four
// 128 x BN x 16 MMAs with both operands in shared memory), measured on GB300 (qkv layer,
// clock64 wait accounting): about 800 + 2.2 BN cycles per block with TMA and the epilogue
// running (1147 / 1272 / 1373 at BN = 160 / 224 / 256).  Each MMA reads A (4 KB) and B
// (32 BN bytes) from shared memory, and the tensor core takes in shared-memory operands at
// about 57 B per cycle, so an MMA costs about (4096 + 32 BN) / 57 cycles rather than BN / 2.
double stage_cycles_a16(int BN) { return 2.0 * (800.0 + 2.2 * BN); }

// Fused path: the decoder warps rebuild BN x 16 groups per stage.  With 8-bit codes
// the stage is bound by shared-memory traffic: per group M codeword lookups of 16 B,
// the 16-byte decoded store and the tensor core's 16-byte read, plus 32 KB of
// activations (TMA write, converter read), at about 80 B per cycle (measured on
// GB300), and by the lookup latency (about 1000 cycles) when there is little work.
// 16-bit codes gather their codewords from L2: about (12 + 12*M) * 2 issue cycles
// per group over the 6 decoder warps (192 threads).
double decode_stage_cycles(int BN, int M, int B) {
  if (B == 16) return BN * 16.0 * (12.0 + 12.0 * M) * 2.0 / 192.0;
  const double bytes = BN * 16.0 * (16.0 * M + 32.0) + 32768.0;
  return std::max(1000.0, bytes / 80.0);
}

int book_smem_bytes(bool fused, int M, int B) {
  return (fused && B == 8) ? M * 256 * 16 * aq::fused_book_copies(M) : 0;
}

// Fused path: packed code bytes of one row for one 64-wide K block, staged per stage.
int code_smem_bytes(bool fused, int M, int B) { return fused ? 8 * M * (B / 8) : 0; }

// fp32 epilogue staging: fp32 output, or split-K partials stored to the workspace
bool plan_f32_staging(const Plan& pl, bool f32_out) {
  return f32_out || (pl.splits > 1 && !pl.cluster);
}

int plan_epi_warps(bool fused, bool f32_staging, int BN) {
  // the dense path has no decoder warps: 8 epilogue warps double the epilogue's rate,
  // which bounds tiles with small K; fp32 staging would cost a pipeline stage
  return (!fused && !f32_staging && BN >= 64) ? 8 : 4;
}

void finish_plan(Plan& pl, bool f32_out, int book_bytes, int code_bytes, bool fused) {
  pl.acc_stride = pl.BN;
  pl.a_col = 2 * pl.acc_stride;
  pl.sb = pl.a16 ? kA16StageBlocks : aq::kStageBlocks;
  const bool f32_staging = plan_f32_staging(pl, f32_out);
  pl.epi_warps = plan_epi_warps(fused, f32_staging, pl.BN);
  pl.stages = aq::gemm_max_stages(pl.BN, f32_staging, book_bytes, code_bytes, pl.epi_warps,
                                  pl.a16 != 0, pl.sb);
  pl.a_stages = pl.a16 ? 0 : aq::gemm_a_stages(pl.BN);
  pl.total_tiles = pl.m_tiles * pl.n_tiles * pl.splits;
}

// Shared-memory bytes of the pipeline ring (where an in-cluster split keeps its fp32
// partial tile of 128 x BN x 4 bytes once the mainloop is done).
size_t ring_bytes(const Plan& pl) {
  const int SB = pl.a16 ? pl.sb : aq::kStageBlocks;
  const size_t a = pl.a16 ? static_cast<size_t>(SB) * aq::kBM * 128 : aq::kStageBlocks * aq::kBM * 64;
  return static_cast<size_t>(pl.stages) * (static_cast<size_t>(SB) * pl.BN * 128 + a);
}

// Picks the N tile and the K split that minimise a model of the busiest SM's time:
// waves x (stage cycles x stages per tile + a fixed tile overhead), plus the cost of
// the split-K reduction when K is split: either the partials' round trip through the
// workspace and the reduce kernel (its launch waits for the GEMM to retire, about
// 2 us), or, when all clusters of S <= 8 CTAs are resident at once, the in-cluster sum
// through distributed shared memory.  Depends only on the shapes (and, for the fused
// path, on the code format).
// Diagnostic plan override of this host thread (aq_set_plan_override): N tile, K
// splits, in-cluster sum (-1: free).  Plans the shapes cannot take are skipped and the
// cost-model plan runs instead.
struct PlanOverride {
  int BN = 0, splits = 0, cluster = -1;
};
thread_local PlanOverride g_plan_override;

// Time after which a pipeline wait of the tensor-core kernels gives up, for this host
// thread's later launches (aq_set_wait_limit_ns; tests of the failure path).
thread_local unsigned long long g_wait_limit_ns = aq::kWaitLimitNs;

// a16: the shared-memory A form (fp16 activations in global memory, dense weights).
Plan plan_gemm(int T, int N, int K, int m_tiles, bool allow_split, bool f32_out,
               bool fused = false, int M = 1, int B = 8, bool a16 = false) {
  const int num_kb = (K + aq::kBK - 1) / aq::kBK;
  const int book_bytes = book_smem_bytes(fused, M, B);
  const int code_bytes = code_smem_bytes(fused, M, B);
  const PlanOverride ov = g_plan_override;
  double best = 1e30;
  Plan bp{};
  // forced: only the override's choices (a cluster plan is then allowed beyond one wave of
  // clusters, which still runs correctly, in waves)
  auto search = [&](bool forced) {
    for (int BN = aq::kMaxBN; BN >= 32; BN -= 32) {
      if (forced && ov.BN > 0 && BN != ov.BN) continue;
      if (!a16 && aq::gemm_a_stages(BN) < 2) continue;
      if (aq::gemm_max_stages(BN, true, book_bytes, code_bytes, 4, a16, kA16StageBlocks) < 2)
        continue;
      const int n_tiles = (N + BN - 1) / BN;
      const int max_split = allow_split ? std::min(num_kb, 64) : 1;
      double st_cyc = a16 ? stage_cycles_a16(BN) : stage_cycles(BN);
      if (fused) st_cyc = std::max(st_cyc, decode_stage_cycles(BN, M, B));
      for (int sp = 1; sp <= max_split; ++sp) {
        const int kbps = (num_kb + sp - 1) / sp;
        const int s_eff = (num_kb + kbps - 1) / kbps;
        if (s_eff != sp) continue;
        if (forced && ov.splits > 0 && s_eff != ov.splits) continue;
        const long tiles = static_cast<long>(m_tiles) * n_tiles * s_eff;
        const long waves = (tiles + kPlanSMs - 1) / kPlanSMs;
        const double tile_cycles = (kbps / 2) * st_cyc + (kbps & 1) * 0.5 * st_cyc + 800.0;
        for (int cl = 0; cl < 2; ++cl) {
          if (forced && ov.cluster >= 0 && cl != ov.cluster) continue;
          // Epilogue: about 900 cycles per 32-column chunk and epilogue warp group (4 warps;
          // 8 on the dense path without fp32 staging).  It overlaps the next tile's
          // mainloop (double-buffered accumulators), so a tile takes the longer of the two,
          // and the last tile's epilogue adds to the end.  The same estimate for every output
          // type keeps the plan, and so the workspace, independent of it.
          const bool partials = s_eff > 1 && !cl;
          const int ew = (!fused && !partials && BN >= 64) ? 8 : 4;
          const double epi = (BN / 32.0) * 900.0 / (ew / 4);
          double t = (static_cast<double>(waves) * std::max(tile_cycles, epi) + epi) / 1.9e9;
          if (cl) {
            if (s_eff < 2 || s_eff > aq::kMaxClusterSplits) continue;
            if (!forced && static_cast<long>(m_tiles) * n_tiles > kPlanMaxClusters[s_eff]) continue;
            if (a16) {
              // the partial tile must fit in the ring
              Plan tp{};
              tp.BN = BN;
              tp.a16 = 1;
              tp.sb = kA16StageBlocks;
              tp.stages = aq::gemm_max_stages(BN, false, 0, 0, plan_epi_warps(false, false, BN),
                                              true, kA16StageBlocks);
              if (ring_bytes(tp) < static_cast<size_t>(aq::kBM) * BN * 4) continue;
            }
            // one tile per CTA; then the partial's shared-memory write, two cluster
            // barriers and the 128 x BN x 4 bytes each CTA reads over distributed shared
            // memory (about 3000 + 8 BN cycles measured on GB300 layers)
            t = (tile_cycles + 3000.0 + 8.0 * BN) / 1.9e9;
          } else if (s_eff > 1) {
            // partials written and read back (mostly from L2) + the reduce kernel
            const double part_bytes = s_eff * 8.0 * T * static_cast<double>(N);
            t += part_bytes / (part_bytes < 64e6 ? 15.0e12 : 6.0e12) + 2.0 * T * N / 6.0e12 +
                 2.0e-6;
          }
          if (t < best * 0.999) {
            best = t;
            bp = Plan{};
            bp.BN = BN;
            bp.n_tiles = n_tiles;
            bp.m_tiles = m_tiles;
            bp.splits = s_eff;
            bp.kb_per_split = kbps;
            bp.num_kb = num_kb;
            bp.cluster = cl;
            bp.a16 = a16 ? 1 : 0;
          }
        }
      }
    }
  };
  if (ov.BN > 0 || ov.splits > 0 || ov.cluster >= 0) search(true);
  if (best > 1e29) search(false);
  finish_plan(bp, f32_out, book_bytes, code_bytes, fused);
  return bp;
}

// The ring must hold an in-cluster split's partial tile (checked when planning; kept as an
// invariant of every plan that runs).
bool plan_ring_ok(const Plan& pl) {
  return !pl.cluster || ring_bytes(pl) >= static_cast<size_t>(aq::kBM) * pl.BN * 4;
}

size_t dense_ws_bytes(int T, int N, int K, const Plan& pl) {
  size_t b = align_up(static_cast<size_t>(N) * K * 2, 1024);
  if (pl.splits > 1 && !pl.cluster) b += align_up(static_cast<size_t>(pl.splits) * T * N * 4, 1024);
  return b;
}

// Fused path workspace: only the split-K partial sums (no decoded weights).
size_t fused_ws_bytes(int T, int N, const Plan& pl) {
  return (pl.splits > 1 && !pl.cluster) ? align_up(static_cast<size_t>(pl.splits) * T * N * 4, 1024)
                                        : 0;
}

// AUTO decodes inside the GEMM (fused path) when every weight tile is decoded by at
// most this many CTAs (one per 128-row M tile); beyond it a separate decode pass
// into the workspace is cheaper.
constexpr int kFusedAutoMaxMTiles = 1;

// Path of a convolution: -1 unknown path, -2 path cannot run this layer.  The
// kernel-aware grouping (g = 9) is decoded by its own pass: dense path only.
int resolve_conv_path(int path, int m_tiles, int g) {
  const bool kaq = g == kKaqGroup;
  switch (path) {
    case AQ_PATH_AUTO:
      return (m_tiles <= kFusedAutoMaxMTiles && !kaq) ? AQ_PATH_FUSED : AQ_PATH_DENSE;
    case AQ_PATH_DENSE:
    case AQ_PATH_PREDECODED:
      return path;
    case AQ_PATH_FUSED:
      return kaq ? -2 : path;
    case AQ_PATH_LUT:
      return -2;
    default:
      return -1;
  }
}

// ---- lookup-table path (linear layers, 8-bit codes, T <= 16)
constexpr int kLutMaxT = 16;       // tokens per call the LUT kernel handles

struct LutPlan {
  int vec, J, Tp, chunks, rows_per_cta, ctas;
  size_t ws_bytes;
};

// lutr_kernel: each CTA takes at least this many 32-row blocks of (chunk, row block) units, so
// that building a chunk's 64 KB of tables is paid for by enough lookups.
constexpr int kLutrMinRowBlocksPerCta = 64;
// The time of one chunk's table build, in 32-row blocks of lookups (measured: a build takes
// about as long as streaming 60-90 row blocks of one CTA).
constexpr int kLutrBuildRowBlocks = 64;

// Contiguous ranges of the chunk-major (chunk, 32-row block) units for `ctas` CTAs such that
// no CTA's cost -- its row blocks plus kLutrBuildRowBlocks per chunk whose tables it builds --
// exceeds `tau`: each CTA in turn takes as many units as that allows.  Fills bounds[0..ctas]
// (later CTAs may get empty ranges) and returns whether every unit was placed.
bool lutr_fill(int64_t units, int64_t nrb, int ctas, int64_t tau, int64_t* bounds) {
  int64_t u = 0;
  bounds[0] = 0;
  for (int b = 0; b < ctas; ++b) {
    int64_t r = u < units ? tau - kLutrBuildRowBlocks : 0;   // the first chunk's build
    while (r > 0 && u < units) {
      const int64_t e = std::min(units, (u / nrb + 1) * nrb);  // end of the current chunk
      if (u + r <= e) {
        u += r;
        r = 0;
      } else {
        r -= e - u;
        u = e;
        r -= kLutrBuildRowBlocks;                            // entering the next chunk
      }
    }
    bounds[b + 1] = u;
  }
  return u >= units;
}

// The smallest such cost for `ctas` CTAs (1 <= ctas <= kLutrMaxCtas), with its ranges in
// bounds: bisection between a cost no split meets (each CTA's share of the units plus one
// build, less one) and one the even split meets (its busiest CTA), so a handful of fills.
// The last few results are kept per host thread, so repeated calls of a layer skip the search.
int64_t lutr_partition(int64_t units, int64_t nrb, int ctas, int64_t* bounds) {
  struct Entry {
    int64_t units = -1, nrb = 0, tau = 0;
    int ctas = 0;
    int64_t b[aq::kLutrMaxCtas + 1];
  };
  thread_local Entry cache[8];
  thread_local int next = 0;
  for (const Entry& e : cache) {
    if (e.units == units && e.nrb == nrb && e.ctas == ctas) {
      std::memcpy(bounds, e.b, sizeof(int64_t) * (ctas + 1));
      return e.tau;
    }
  }
  int64_t hi = 0;
  for (int b = 0; b < ctas; ++b) {
    const int64_t u0 = units * b / ctas, u1 = units * (b + 1) / ctas;
    if (u1 > u0)
      hi = std::max(hi, u1 - u0 + kLutrBuildRowBlocks * ((u1 - 1) / nrb - u0 / nrb + 1));
  }
  int64_t lo = (units + ctas - 1) / ctas + kLutrBuildRowBlocks - 1;
  while (lo + 1 < hi) {
    const int64_t mid = lo + (hi - lo) / 2;
    if (lutr_fill(units, nrb, ctas, mid, bounds))
      hi = mid;
    else
      lo = mid;
  }
  lutr_fill(units, nrb, ctas, hi, bounds);
  Entry& e = cache[next];
  next = (next + 1) % 8;
  e.units = units;
  e.nrb = nrb;
  e.ctas = ctas;
  e.tau = hi;
  std::memcpy(e.b, bounds, sizeof(int64_t) * (ctas + 1));
  return hi;
}

LutPlan plan_lut(int T, int K, int N, int M) {
  LutPlan lp{};
  const bool mm = M == 1 || M == 2 || M == 4;
  if (T <= 4 && mm) {
    // lutr_kernel: TP = 1, 2 or 4 floats per entry; a chunk is 32 / TP code bytes of every row
    // (32 / (TP * M) groups); one CTA of 1024 threads per SM at most, each with a contiguous
    // range of (chunk, 32-row block) units (lutr_partition, at launch)
    lp.vec = 2;
    lp.Tp = T == 1 ? 1 : (T == 2 ? 2 : 4);
    const int KB = (K + 63) / 64;
    const int nt = 32 / lp.Tp;
    lp.J = nt / M;
    lp.chunks = (KB * 8 * M + nt - 1) / nt;
    const int64_t nrb = (N + 31) / 32;
    const int64_t units = static_cast<int64_t>(lp.chunks) * nrb;
    lp.ctas = static_cast<int>(std::max<int64_t>(
        1, std::min<int64_t>(kPlanSMs, units / kLutrMinRowBlocksPerCta)));
    // fewer CTAs, a whole multiple of the chunks, when no CTA then builds two chunks' tables and
    // the busiest CTA's cost comes out lower
    if (lp.chunks <= lp.ctas) {
      const int aligned = lp.ctas / lp.chunks * lp.chunks;
      int64_t b[kPlanSMs + 1];
      if (aligned < lp.ctas &&
          lutr_partition(units, nrb, aligned, b) < lutr_partition(units, nrb, lp.ctas, b))
        lp.ctas = aligned;
    }
    lp.rows_per_cta = 0;
    lp.ws_bytes = align_up(static_cast<size_t>(lp.chunks) * T * N * 4, 1024);
    return lp;
  }
  if (T == 1) {
    // lutv_kernel (one token, M other than 1, 2, 4): chunks of whole packed K blocks (two for
    // M <= 4, else one: at most 64 KB of tables), over (chunk, row slice) CTAs -- as many row
    // slices as keep them within one wave (a second, nearly empty wave would double the time)
    lp.vec = 1;
    lp.Tp = 1;
    lp.J = 8 * (M <= 4 ? 2 : 1);
    const int G = K / 8;
    lp.chunks = (G + lp.J - 1) / lp.J;
    const size_t smem = static_cast<size_t>(lp.J) * M * 256 * 4 + static_cast<size_t>(lp.J) * 8 * 4;
    const int per_sm = std::max(1, std::min(3, static_cast<int>(232448 / (smem + 1024))));
    int n_slices = per_sm * kPlanSMs / lp.chunks;
    if (n_slices < 1) n_slices = 1;
    lp.rows_per_cta = ((N + n_slices - 1) / n_slices + 31) / 32 * 32;
    lp.ws_bytes = align_up(static_cast<size_t>(lp.chunks) * N * 4, 1024);
    return lp;
  }
  lp.Tp = T <= 4 ? 4 : (T <= 8 ? 8 : 16);
  lp.J = 8;
  while (lp.J > 1 && static_cast<size_t>(lp.J) * M * 256 * lp.Tp * 4 > 160 * 1024) lp.J >>= 1;
  const int G = K / 8;
  lp.chunks = (G + lp.J - 1) / lp.J;
  int n_slices = (2 * kPlanSMs + lp.chunks - 1) / lp.chunks;
  if (n_slices < 1) n_slices = 1;
  lp.rows_per_cta = ((N + n_slices - 1) / n_slices + 31) / 32 * 32;
  lp.ws_bytes = align_up(static_cast<size_t>(lp.chunks) * T * N * 4, 1024);
  return lp;
}

// Few-token path: linear layers up to this many tokens; AUTO takes it up to
// kFewTokensAutoMaxT (measured on GB300: faster than the table and fused paths at
// T <= 4, equal at 8, slower at 16).
constexpr int kFewTokensMaxT = 16;
constexpr int kFewTokensAutoMaxT = 4;

// AUTO / explicit path of a linear layer: -1 unknown path, -2 path cannot run this layer.
// AUTO takes the table path (lutr_kernel for up to four tokens with M = 1, 2 or 4; lutv_kernel
// for one token with other M) from this many bytes of 8-bit codes, the few-token kernel below.
// Measured on GB300 (layer only, graph replay over 4 rotating layers, us, table / few-token):
// T=1 2x8 33.6 MB 19.1 / 44.9, 8.4 MB 8.8-9.2 / 12.4-13.3, 4.2 MB 8.7 / 8.2-8.8, 0.7 MB
// 10.3 / 4.1; T=2 2x8 33.6 MB 23.8 / 62.0, 8.4 MB 12.8-14.3 / 17.4-17.5, 4.2 MB 9.2 / 9.8;
// T=4 2x8 33.6 MB 44.5 / 126.5, 4.2 MB 12.8 / 14.4; T=1 1x8 16.8 MB 13.3 / 33.5; T=1 4x8
// 67.1 MB 36.4 / 198; T=4 4x8 67.1 MB 101 / 283.
constexpr size_t kLutAutoMinCodeBytes = 6u << 20;

int resolve_linear_path(int path, int T, int B, int N = 0, int K = 0, int M = 0) {
  const int m_tiles = (T + aq::kBM - 1) / aq::kBM;
  switch (path) {
    case AQ_PATH_AUTO:
      if (T <= kFewTokensAutoMaxT && B == 8 && (T == 1 || M == 1 || M == 2 || M == 4) &&
          static_cast<size_t>(N) * (K / 8) * M >= kLutAutoMinCodeBytes)
        return AQ_PATH_LUT;
      if (T <= kFewTokensAutoMaxT) return AQ_PATH_FEW_TOKENS;
      return m_tiles <= kFusedAutoMaxMTiles ? AQ_PATH_FUSED : AQ_PATH_DENSE;
    case AQ_PATH_FEW_TOKENS:
      return T <= kFewTokensMaxT ? path : -2;
    case AQ_PATH_DENSE:
    case AQ_PATH_FUSED:
    case AQ_PATH_PREDECODED:
      return path;
    case AQ_PATH_LUT:
      return (B == 8 && T <= kLutMaxT) ? AQ_PATH_LUT : -2;
    default:
      return -1;
  }
}

int path_error(int rp, int path) {
  if (rp == -2)
    return set_error(AQ_ERR_UNSUPPORTED,
                     "path %d cannot run this layer (the table path is for linear layers with "
                     "8-bit codes and T <= %d)",
                     path, kLutMaxT);
  return set_error(AQ_ERR_UNSUPPORTED, "path %d not available", path);
}

// Conv tile geometry: 128 output pixels per tile as one 4-D box.
struct ConvGeom {
  int Ho, Wo, tiles_per_img, rows_per_tile, imgs_per_tile, m_tiles, bw, bh, bn;
};

int conv_geometry(int Nb, int H, int W, int kh, int kw, int stride, int pad, ConvGeom* g) {
  g->Ho = (H + 2 * pad - kh) / stride + 1;
  g->Wo = (W + 2 * pad - kw) / stride + 1;
  const int Wo = g->Wo, Ho = g->Ho;
  if (stride * Wo > 256) return set_error(AQ_ERR_UNSUPPORTED, "conv output width %d too wide", Wo);
  if (Wo > aq::kBM || aq::kBM % Wo != 0)
    return set_error(AQ_ERR_UNSUPPORTED, "conv output width %d must divide 128", Wo);
  const int rpt = aq::kBM / Wo;
  if (rpt <= Ho) {
    if (Ho % rpt != 0)
      return set_error(AQ_ERR_UNSUPPORTED, "conv output height %d not a multiple of %d", Ho, rpt);
    g->rows_per_tile = rpt;
    g->tiles_per_img = Ho / rpt;
    g->imgs_per_tile = 0;
    g->m_tiles = Nb * g->tiles_per_img;
    g->bw = Wo;
    g->bh = rpt;
    g->bn = 1;
  } else {
    if (rpt % Ho != 0)
      return set_error(AQ_ERR_UNSUPPORTED, "conv image %dx%d does not tile 128 pixels", Ho, Wo);
    g->imgs_per_tile = rpt / Ho;
    g->rows_per_tile = Ho;
    g->tiles_per_img = 1;
    g->m_tiles = (Nb + g->imgs_per_tile - 1) / g->imgs_per_tile;
    g->bw = Wo;
    g->bh = Ho;
    g->bn = g->imgs_per_tile;
  }
  return AQ_OK;
}

int check_conv_args(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride,
                    int pad) {
  if (Nb < 0 || H <= 0 || W <= 0 || Cin <= 0 || Cout <= 0)
    return set_error(AQ_ERR_SHAPE, "conv sizes must be positive (Nb >= 0)");
  if (kh != 3 || kw != 3 || pad != 1)
    return set_error(AQ_ERR_UNSUPPORTED, "only 3x3 convolutions with pad 1 are supported");
  if (stride != 1 && stride != 2) return set_error(AQ_ERR_UNSUPPORTED, "stride must be 1 or 2");
  if (Cin % 64 != 0) return set_error(AQ_ERR_UNSUPPORTED, "Cin=%d must be a multiple of 64", Cin);
  if (Cout % 8 != 0) return set_error(AQ_ERR_SHAPE, "Cout=%d must be a multiple of 8", Cout);
  return AQ_OK;
}


// ---- kernel timing (aq_profile_*): CUDA event pairs around each launch
namespace prof {
std::mutex mu;
std::atomic<bool> enabled{false};
struct Rec {
  cudaEvent_t a, b;
  int kind;
};
std::vector<Rec> pending;
std::vector<cudaEvent_t> pool;
double ms[AQ_PROFILE_KINDS] = {};
int64_t launches[AQ_PROFILE_KINDS] = {};

cudaEvent_t take_locked() {
  if (!pool.empty()) {
    cudaEvent_t e = pool.back();
    pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

void fold_locked(bool accumulate) {
  for (const Rec& r : pending) {
    float t = 0.0f;
    if (cudaEventSynchronize(r.b) == cudaSuccess && cudaEventElapsedTime(&t, r.a, r.b) == cudaSuccess) {
      if (accumulate) {
        ms[r.kind] += t;
        launches[r.kind] += 1;
      }
    } else {
      (void)cudaGetLastError();  // do not leave the failure for the next launch check
    }
    pool.push_back(r.a);
    pool.push_back(r.b);
  }
  pending.clear();
}
}  // namespace prof

// Records an event pair around the launches made while it is alive.  Under stream
// capture the records become external event-record nodes of the graph, so each
// replay of the graph stamps them again (the last replay is what a read sees).
cudaError_t record_event(cudaEvent_t e, cudaStream_t st) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
    return cudaEventRecordWithFlags(e, st, cudaEventRecordExternal);
  return cudaEventRecord(e, st);
}

struct ProfScope {
  cudaStream_t st;
  int kind;
  cudaEvent_t a = nullptr;
  ProfScope(int k, cudaStream_t s) : st(s), kind(k) {
    if (!prof::enabled.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> g(prof::mu);
    a = prof::take_locked();
    if (a && record_event(a, st) != cudaSuccess) {
      (void)cudaGetLastError();
      prof::pool.push_back(a);
      a = nullptr;
    }
  }
  ~ProfScope() {
    if (!a) return;
    std::lock_guard<std::mutex> g(prof::mu);
    cudaEvent_t b = prof::take_locked();
    if (!b || record_event(b, st) != cudaSuccess) {
      (void)cudaGetLastError();
      prof::pool.push_back(a);
      if (b) prof::pool.push_back(b);
      return;
    }
    prof::pending.push_back({a, b, kind});
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (prof::pending.size() > 16384 && cudaStreamIsCapturing(st, &cs) == cudaSuccess &&
        cs == cudaStreamCaptureStatusNone)
      prof::fold_locked(true);
  }
};

enum ProfKind { kProfQuant = 0, kProfPack = 1, kProfDecode = 2, kProfGemm = 3, kProfSplitK = 4,
                kProfLutBuild = 5, kProfLutGather = 6, kProfFused = 7 };

int sm_count() {
  static int counts[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    (void)cudaGetLastError();
    return kPlanSMs;
  }
  if (counts[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
      (void)cudaGetLastError();
      n = kPlanSMs;
    }
    counts[dev] = n;
  }
  return counts[dev];
}

// Dense path after the activation map is built: decode W-hat into the workspace,
// then the tensor-core GEMM with the fused epilogue (or split-K partials + reduce).
// Tensor-core path after the activation map is built.  Dense: decode W-hat into the
// workspace (Wdec), then the GEMM streams it with TMA.  Fused (Wdec == nullptr): the
// GEMM's decoder warps rebuild each weight tile in shared memory from the codes.
// kaq: the codes use the kernel-aware grouping (g = 9, dense path only).
// x16 != nullptr: the layer's fp16 activations, quantized here into the GEMM's int8
// operand xq (the memory mapA points at) with the rule of aq_quant_act and scale p.s_x.
// pl.a16: mapA describes fp16 activations (the 8-bit codes as fp16 integers); with x16 the
// quantizer writes them (into xq, then an fp16 buffer) with the same rule.
int run_gemm(const CUtensorMap& mapA, aq::GemmParams p, const Plan& pl, const void* codes_packed,
             const void* codebooks, int M, int B, void* Wdec, float* partial, cudaStream_t st,
             bool kaq = false, const void* x16 = nullptr, int8_t* xq = nullptr,
             bool predecoded = false, int64_t x_elems = 0) {
  const bool fused = Wdec == nullptr;
  if (!plan_ring_ok(pl)) return set_error(AQ_ERR_UNSUPPORTED, "plan: partial tile exceeds the ring");
  p.fused = fused ? 1 : 0;
  p.a16 = pl.a16;
  p.sb = pl.sb;
  p.wait_ns = g_wait_limit_ns;
  p.codes = codes_packed;
  p.books = codebooks;
  p.M = M;
  p.B = B;
  p.book_bytes = book_smem_bytes(fused, M, B);
  p.BN = pl.BN;
  p.num_kb = pl.num_kb;
  p.kb_per_split = pl.kb_per_split;
  p.m_tiles = pl.m_tiles;
  p.n_tiles = pl.n_tiles;
  p.splits = pl.splits;
  p.total_tiles = pl.total_tiles;
  p.stages = pl.stages;
  p.a_stages = pl.a_stages;
  p.acc_stride = pl.acc_stride;
  p.a_col = pl.a_col;
  p.cluster = pl.cluster;
  p.epi_warps = pl.epi_warps;
  // The shared-memory A form takes 12 epilogue warps (three per TMEM lane quarter) where the
  // epilogue, not the mainloop, bounds a tile -- the 8-bit activation rule of the _q8 / _ex
  // code outputs costs about four times the fp16 epilogue's instructions per value, and a tile
  // of at most 8 K blocks has a shorter mainloop than its epilogue -- when the extra staging
  // costs no pipeline stage.  Measured on GB300 (T=65536, K=384, N=1152, N tile 256, 8 warps):
  // fp16 output 66 us, int8 codes 110 us.
  // (8 epilogue warps imply fp16 / int8 staging: no fp32 output, no partials)
  if (pl.a16 && !fused && !pl.cluster && pl.epi_warps == 8 &&
      (p.out_q8 || pl.kb_per_split <= 8) &&
      aq::gemm_max_stages(pl.BN, false, 0, 0, 12, true, pl.sb) >= pl.stages)
    p.epi_warps = 12;
  p.partial = (pl.splits > 1 && !pl.cluster) ? partial : nullptr;
  const int T = p.T, N = p.N, K = p.K;
  int r;
  CUtensorMap mapB, mapY;
  std::memset(&mapB, 0, sizeof(mapB));
  if (!fused) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(N)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(aq::kBK), static_cast<cuuint32_t>(pl.BN)};
    r = encode(&mapB, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, Wdec, dims, strides, box,
               CU_TENSOR_MAP_SWIZZLE_128B);
    if (r) return r;
  }
  if (p.partial) {
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(T),
                          static_cast<cuuint64_t>(pl.splits)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(N) * 4, static_cast<cuuint64_t>(T) * N * 4};
    cuuint32_t box[3] = {32, 32, 1};
    r = encode(&mapY, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, p.partial, dims, strides, box,
               CU_TENSOR_MAP_SWIZZLE_128B);
  } else if (p.out_q8 == aq::kOutCodesI8) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(T)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(N)};
    cuuint32_t box[2] = {32, 32};
    r = encode(&mapY, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, p.y, dims, strides, box,
               CU_TENSOR_MAP_SWIZZLE_NONE);
  } else if (p.out_f32) {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(T)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(N) * 4};
    cuuint32_t box[2] = {32, 32};
    r = encode(&mapY, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, p.y, dims, strides, box,
               CU_TENSOR_MAP_SWIZZLE_128B);
  } else {
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(T)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(N) * 2};
    cuuint32_t box[2] = {32, 32};
    r = encode(&mapY, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, p.y, dims, strides, box,
               CU_TENSOR_MAP_SWIZZLE_64B);
  }
  if (r) return r;
  cudaError_t e;
  // the activation tensor x16 quantized into xq: T x K for a linear layer; the caller gives the
  // input tensor's size for a convolution (T, K there are output pixels and 9 * Cin)
  if (x_elems == 0) x_elems = static_cast<int64_t>(T) * K;
  if (x16) {
    ProfScope ps(kProfQuant, st);
    e = pl.a16 ? aq::launch_quant_act_f16(x16, reinterpret_cast<__half*>(xq), x_elems, p.s_x, st)
               : aq::launch_quant_act(x16, xq, x_elems, p.s_x, st);
    if (e != cudaSuccess) return cuda_status(e, "quantizer launch");
  }
  if (!fused && !predecoded) {
    ProfScope ps(kProfDecode, st);
    e = kaq ? aq::launch_decode_kaq(codes_packed, codebooks, Wdec, N, K / kKaqGroup, M, B, st)
            : aq::launch_decode(codes_packed, codebooks, Wdec, N, K, M, B, st);
    if (e != cudaSuccess) return cuda_status(e, "decode launch");
  }
  {
    ProfScope ps(fused ? kProfFused : kProfGemm, st);
    // in-cluster split-K runs one CTA per (tile, split); otherwise a persistent grid
    const int grid = pl.cluster ? pl.total_tiles : std::min(pl.total_tiles, sm_count());
    e = aq::launch_gemm(mapA, mapB, mapY, p, grid, st);
  }
  if (e != cudaSuccess) return cuda_status(e, "gemm launch");
  if (pl.splits > 1 && !pl.cluster) {
    ProfScope ps(kProfSplitK, st);
    e = aq::launch_splitk_reduce(p, pl.splits, st);
    if (e != cudaSuccess) return cuda_status(e, "split-K reduce launch");
  }
  return ok();
}

// Plan and workspace layout of a tensor-core call on the dense or the fused path.
struct Route {
  bool fused;
  bool predecoded;  // the workspace already holds W-hat: the GEMM only
  Plan pl;
  size_t ws;
};

// a16: fp16 activations (the shared-memory A form) on the dense / predecoded paths.
Route route_gemm(int rp, int T, int N, int K, int m_tiles, bool f32_out, int M, int B,
                 bool a16 = false) {
  Route rt;
  rt.fused = rp == AQ_PATH_FUSED;
  rt.predecoded = rp == AQ_PATH_PREDECODED;
  rt.pl = plan_gemm(T, N, K, m_tiles, true, f32_out, rt.fused, M, B, a16 && !rt.fused);
  rt.ws = rt.fused ? fused_ws_bytes(T, N, rt.pl) : dense_ws_bytes(T, N, K, rt.pl);
  return rt;
}

// Activations of a layer call: int8 codes (aq_linear, aq_conv2d_nhwc), fp16 activations this
// call quantizes (aq_linear_f16, aq_conv2d_nhwc_f16), or the codes already held as fp16 values
// (aq_linear_a16).
enum ActKind { kActInt8 = 0, kActF16 = 1, kActF16Codes = 2 };

// The tensor-core form of a layer on the dense paths.  The shared-memory A form (fp16 A) takes N
// tiles up to 256 wide but each of its MMAs costs at least ~138 cycles (128 x N x 16, measured);
// the tensor-memory A form (int8 codes converted into tensor memory) takes N tiles up to 192.  A
// call that quantizes fp16 activations itself writes fp16 codes only when the fp16 form's plan
// has no K split and a wider N tile than the int8 form's plan; codes given as fp16 always take
// it.  Measured on GB300 (GEMM alone, weights decoded beforehand, us int8 / fp16 form): qkv
// 4096 x 960 x 2880 28.1 / 25.1 (N tiles 160 / 224); 8192 x 576 x 1728 24.0 / 21.9 (192 / 256);
// 16384 x 192 x 576 18.0 / 14.5 (96 / 192); 2048 x 960 x 2880 16.8 / 17.3 (160 / 160);
// 2048 x 960 x 960 9.5 / 15.1 (fp16 plan split 2); the 64x64 W4A8 3x3 conv, whole call,
// 54.7 / 60.9 (192 / 192).
Route route_layer(int rp, int T, int N, int K, int m_tiles, bool f32_out, int M, int B,
                  ActKind act) {
  const bool dense = rp == AQ_PATH_DENSE || rp == AQ_PATH_PREDECODED;
  if (act == kActInt8 || !dense) return route_gemm(rp, T, N, K, m_tiles, f32_out, M, B, false);
  const Route r16 = route_gemm(rp, T, N, K, m_tiles, f32_out, M, B, true);
  // (a plan override wider than the int8 form's widest tile can only mean the fp16 form)
  if (act == kActF16Codes || g_plan_override.BN > aq::kA8MaxBN) return r16;
  const Route r8 = route_gemm(rp, T, N, K, m_tiles, f32_out, M, B, false);
  return (r16.pl.splits == 1 && r16.pl.BN > r8.pl.BN) ? r16 : r8;
}

int check_workspace(const void* workspace, size_t workspace_bytes, size_t need) {
  if (need == 0) return AQ_OK;
  if (!workspace || workspace_bytes < need || !aligned16(workspace))
    return set_error(AQ_ERR_WORKSPACE, "workspace needs %zu bytes (got %zu)", need, workspace_bytes);
  return AQ_OK;
}

// Dense: [decoded W-hat fp16 (N x K)][split-K partials]; fused: [split-K partials].
void ws_pointers(const Route& rt, void* workspace, int N, int K, void** Wdec, float** partial) {
  if (rt.fused) {
    *Wdec = nullptr;
    *partial = static_cast<float*>(workspace);
  } else {
    *Wdec = workspace;
    *partial = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) +
                                        align_up(static_cast<size_t>(N) * K * 2, 1024));
  }
}

int encode_linear_a(CUtensorMap* mapA, const int8_t* xq, int T, int K) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(T)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(K)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(aq::kBK), static_cast<cuuint32_t>(aq::kBM)};
  return encode(mapA, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, xq, dims, strides, box,
                CU_TENSOR_MAP_SWIZZLE_64B);
}

// fp16 activations [T][K] for the shared-memory A form: 64 x 128 boxes, 128-byte swizzle
// (the layout of the weight boxes).
int encode_linear_a16(CUtensorMap* mapA, const void* xh, int T, int K) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(T)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(aq::kBK), static_cast<cuuint32_t>(aq::kBM)};
  return encode(mapA, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, xh, dims, strides, box,
                CU_TENSOR_MAP_SWIZZLE_128B);
}

// GemmParams::out_q8 / SkinnyParams::out_q8 of an output dtype.
int out_codes(int out_dtype) {
  return out_dtype == AQ_DTYPE_I8 ? aq::kOutCodesI8
                                  : (out_dtype == AQ_DTYPE_F16_CODES ? aq::kOutCodesF16 : 0);
}

// Output kinds of the layer entry points: AQ_DTYPE_F16 / AQ_DTYPE_F32 through
// aq_linear / aq_conv2d_nhwc, AQ_DTYPE_I8 (quantized with s_out) through the _q8
// variants.  int8 rows need N % 16 == 0 (16-byte TMA row stride).
int check_output(int out_dtype, float s_out, int N) {
  if (out_dtype == AQ_DTYPE_I8 || out_dtype == AQ_DTYPE_F16_CODES) {
    if (!(s_out > 0.0f) || s_out == __builtin_inff())
      return set_error(AQ_ERR_SHAPE, "s_out must be finite and > 0");
    if (out_dtype == AQ_DTYPE_I8 && N % 16 != 0)
      return set_error(AQ_ERR_SHAPE, "int8 output needs N %% 16 == 0");
    return AQ_OK;
  }
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d", out_dtype);
  return AQ_OK;
}

int linear_impl(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
                const void* scale, const void* bias, void* y, int out_dtype, float s_out, int T,
                int K, int N, int g, int M, int B, void* workspace, size_t workspace_bytes,
                int path, void* stream, const void* x16 = nullptr, const void* xh = nullptr);
int linear_ws(int T, int K, int N, int g, int M, int B, int path, ActKind act, size_t* bytes);

// Path of aq_linear_a16 (fp16 activations): the dense tensor-core paths only.
int resolve_a16_path(int path) {
  if (path == AQ_PATH_AUTO) return AQ_PATH_DENSE;
  if (path == AQ_PATH_DENSE || path == AQ_PATH_PREDECODED) return path;
  return -2;
}
int conv_impl(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
              const void* scale, const void* bias, void* y, int out_dtype, float s_out, int Nb,
              int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g, int M,
              int B, void* workspace, size_t workspace_bytes, int path, void* stream,
              const void* x16 = nullptr, const void* xh = nullptr);
int conv_ws(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g,
            int M, int B, int path, ActKind act, size_t* bytes);

}  // namespace

extern "C" {

int aq_abi_version(void) { return AQ_ABI_VERSION; }

int aq_profile_enable(int on) {
  std::lock_guard<std::mutex> g(prof::mu);
  prof::fold_locked(false);
  for (int i = 0; i < AQ_PROFILE_KINDS; ++i) {
    prof::ms[i] = 0.0;
    prof::launches[i] = 0;
  }
  prof::enabled.store(on != 0);
  return ok();
}

int aq_profile_read(double* ms_out, int64_t* launches_out, int n_kinds) {
  if (!ms_out || !launches_out) return set_error(AQ_ERR_NULL, "NULL output");
  std::lock_guard<std::mutex> g(prof::mu);
  prof::fold_locked(true);
  for (int i = 0; i < n_kinds; ++i) {
    ms_out[i] = i < AQ_PROFILE_KINDS ? prof::ms[i] : 0.0;
    launches_out[i] = i < AQ_PROFILE_KINDS ? prof::launches[i] : 0;
  }
  return ok();
}

const char* aq_last_error_string(void) { return g_last_error.c_str(); }

int aq_device_error(int* code_out) {
  if (!code_out) return set_error(AQ_ERR_NULL, "code_out is NULL");
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_status(e, "cudaDeviceSynchronize");
  unsigned v = 0;
  e = aq::read_clear_gemm_error(&v);
  if (e != cudaSuccess) return cuda_status(e, "reading device error word");
  unsigned vl = 0;
  e = aq::read_clear_lut_error(&vl);
  if (e != cudaSuccess) return cuda_status(e, "reading device error word");
  v |= vl;
  *code_out = static_cast<int>(v);
  return ok();
}

int aq_packed_size(int N, int K, int g, int M, int B, size_t* bytes) {
  if (!bytes) return set_error(AQ_ERR_NULL, "bytes is NULL");
  int r = check_format(g, M, B, true);
  if (r) return r;
  if (N <= 0 || K <= 0 || K % g != 0) return set_error(AQ_ERR_SHAPE, "need N, K > 0 and K %% g == 0");
  if (g == kKaqGroup)
    *bytes = static_cast<size_t>(N) * (K / g) * M * (B / 8);   // the canonical layout
  else
    *bytes = static_cast<size_t>((K + 63) / 64) * N * (64 / g) * M * (B / 8);
  return ok();
}

int aq_pack(const void* codes_canon, void* codes_packed, int N, int K, int g, int M, int B,
            void* stream) {
  if (!codes_canon || !codes_packed) return set_error(AQ_ERR_NULL, "NULL code buffer");
  int r = check_format(g, M, B, true);
  if (r) return r;
  if (N <= 0 || K <= 0 || K % g != 0) return set_error(AQ_ERR_SHAPE, "need N, K > 0 and K %% g == 0");
  if (!aligned16(codes_canon) || !aligned16(codes_packed))
    return set_error(AQ_ERR_ALIGN, "code buffers must be 16-byte aligned");
  ProfScope ps(kProfPack, static_cast<cudaStream_t>(stream));
  if (g == kKaqGroup) {
    // one group per filter: the decode reads a group's M codes at once, so the
    // stored layout is the canonical [N][Cin][M] itself
    const size_t bytes = static_cast<size_t>(N) * (K / g) * M * (B / 8);
    return cuda_status(cudaMemcpyAsync(codes_packed, codes_canon, bytes, cudaMemcpyDeviceToDevice,
                                       static_cast<cudaStream_t>(stream)),
                       "aq_pack copy");
  }
  return cuda_status(aq::launch_pack(codes_canon, codes_packed, N, K, M, B,
                                     static_cast<cudaStream_t>(stream)),
                     "aq_pack launch");
}

int aq_decode(const void* codes_packed, const void* codebooks, void* W_out, int N, int K, int g,
              int M, int B, void* stream) {
  if (!codes_packed || !codebooks || !W_out) return set_error(AQ_ERR_NULL, "NULL argument");
  int r = check_format(g, M, B, true);
  if (r) return r;
  if (N <= 0 || K <= 0 || K % g != 0) return set_error(AQ_ERR_SHAPE, "need N, K > 0 and K %% g == 0");
  if (!aligned16(codes_packed) || !aligned16(codebooks) || !aligned16(W_out))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  ProfScope ps(kProfDecode, static_cast<cudaStream_t>(stream));
  if (g == kKaqGroup)
    return cuda_status(aq::launch_decode_kaq(codes_packed, codebooks, W_out, N, K / g, M, B,
                                             static_cast<cudaStream_t>(stream)),
                       "aq_decode launch");
  return cuda_status(aq::launch_decode(codes_packed, codebooks, W_out, N, K, M, B,
                                       static_cast<cudaStream_t>(stream)),
                     "aq_decode launch");
}

int aq_codebook_grad(const void* codes_packed, const float* G, const void* scale, float s_x,
                     float* dC, int N, int K, int g, int M, int B, void* stream) {
  int r = check_format(g, M, B, true);
  if (r) return r;
  if (N <= 0 || K <= 0 || K % g != 0) return set_error(AQ_ERR_SHAPE, "need N, K > 0 and K %% g == 0");
  if (!(s_x == s_x) || s_x == __builtin_inff() || s_x == -__builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite");
  if (!codes_packed || !G || !dC) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(codes_packed) || !aligned16(G) || !aligned16(dC) || (scale && !aligned16(scale)))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return cuda_status(aq::launch_codebook_grad(codes_packed, G, static_cast<const __half*>(scale),
                                              s_x, dC, N, K, g, M, B, st),
                     "aq_codebook_grad launch");
}

int aq_code_update(const float* W, const void* codebooks, void* codes, const float* H,
                   int m_first, int m_count, int N, int K, int g, int M, int B, void* stream) {
  int r = check_format(g, M, B);
  if (r) return r;
  if (B != 8) return set_error(AQ_ERR_UNSUPPORTED, "code search supports 8-bit codes only");
  if (N <= 0 || K <= 0 || K % g != 0) return set_error(AQ_ERR_SHAPE, "need N, K > 0 and K %% g == 0");
  if (m_first < 0 || m_count < 0 || m_first + m_count > M)
    return set_error(AQ_ERR_SHAPE, "codebook range [%d, %d) outside [0, %d)", m_first,
                     m_first + m_count, M);
  if (!W || !codebooks || !codes) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(W) || !aligned16(codebooks) || !aligned16(codes) || (H && !aligned16(H)))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  if (m_count == 0) return ok();
  return cuda_status(aq::launch_code_update(W, codebooks, codes, H, m_first, m_count, N, K, M,
                                            static_cast<cudaStream_t>(stream)),
                     "aq_code_update launch");
}

int aq_quant_act(const void* x, int8_t* xq, int64_t numel, float s_x, void* stream) {
  if (numel < 0) return set_error(AQ_ERR_SHAPE, "numel < 0");
  if (!(s_x > 0.0f) || s_x == __builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite and > 0");
  if (numel == 0) return ok();
  if (!x || !xq) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(x) || !aligned16(xq)) return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  ProfScope ps(kProfQuant, static_cast<cudaStream_t>(stream));
  return cuda_status(aq::launch_quant_act(x, xq, numel, s_x, static_cast<cudaStream_t>(stream)),
                     "aq_quant_act launch");
}

int aq_linear_workspace_size(int T, int K, int N, int g, int M, int B, int path, size_t* bytes) {
  return linear_ws(T, K, N, g, M, B, path, kActInt8, bytes);
}

namespace {
// info[0] = resolved path, then for the tensor-core paths [1] BN, [2] K splits,
// [3] in-cluster split sum (0/1), [4] pipeline stages, [5] (tile, split) work items,
// [6] 1 when the MMA reads fp16 activations from shared memory (0: int8 activations
// converted by warps into tensor memory), [7] 64-wide K blocks per pipeline stage.
constexpr int kPlanInfo = 8;
int fill_plan_info(int rp, const Plan* pl, int* info, int n_info) {
  if (!info || n_info < 1) return set_error(AQ_ERR_NULL, "info is NULL or n_info < 1");
  int v[kPlanInfo] = {rp, 0, 0, 0, 0, 0, 0, 0};
  if (pl) {
    v[1] = pl->BN;
    v[2] = pl->splits;
    v[3] = pl->cluster;
    v[4] = pl->stages;
    v[5] = pl->total_tiles;
    v[6] = pl->a16;
    v[7] = pl->sb;
  }
  for (int i = 0; i < n_info; ++i) info[i] = i < kPlanInfo ? v[i] : 0;
  return ok();
}
}  // namespace

int aq_set_plan_override(int BN, int splits, int cluster) {
  if (BN < 0 || BN > aq::kMaxBN || BN % 32 != 0 || splits < 0 || cluster < -1 || cluster > 1)
    return set_error(AQ_ERR_SHAPE, "plan override: BN in {0, 32, ..., %d}, splits >= 0, "
                     "cluster in {-1, 0, 1}", aq::kMaxBN);
  g_plan_override.BN = BN;
  g_plan_override.splits = splits;
  g_plan_override.cluster = cluster;
  return ok();
}

namespace {
// Plan of a linear call; a16: the call has fp16 activations (aq_linear_f16 / aq_linear_a16),
// a16_only: aq_linear_a16 (dense paths only).
int linear_plan_impl(int T, int K, int N, int g, int M, int B, int path, bool a16,
                     bool a16_only, int* info, int n_info) {
  int r = check_format(g, M, B);
  if (r) return r;
  if (T < 0 || N <= 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and N, K > 0");
  if (K % 16 != 0 || N % 8 != 0) return set_error(AQ_ERR_SHAPE, "need K %% 16 == 0 and N %% 8 == 0");
  const int rp = a16_only ? resolve_a16_path(path) : resolve_linear_path(path, T, B, N, K, M);
  if (rp < 0) return path_error(rp, path);
  if (rp == AQ_PATH_LUT) {
    // the table path: [2] chunks (partial sums per output), [5] CTAs of the table kernel
    const LutPlan lp = plan_lut(std::max(T, 1), K, N, M);
    const int r2 = fill_plan_info(rp, nullptr, info, n_info);
    if (r2 == AQ_OK && n_info > 2) info[2] = lp.chunks;
    if (r2 == AQ_OK && n_info > 5) info[5] = lp.vec == 2 ? lp.ctas : 0;
    return r2;
  }
  if (rp == AQ_PATH_FEW_TOKENS) return fill_plan_info(rp, nullptr, info, n_info);
  const Route rt = route_layer(rp, T, N, K, (T + aq::kBM - 1) / aq::kBM, false, M, B,
                              a16_only ? kActF16Codes : (a16 ? kActF16 : kActInt8));
  return fill_plan_info(rp, &rt.pl, info, n_info);
}
}  // namespace

int aq_set_wait_limit_ns(int64_t ns) {
  g_wait_limit_ns = ns < 0 ? aq::kWaitLimitNs : static_cast<unsigned long long>(ns);
  return ok();
}

int aq_linear_plan(int T, int K, int N, int g, int M, int B, int path, int* info, int n_info) {
  return linear_plan_impl(T, K, N, g, M, B, path, false, false, info, n_info);
}

int aq_linear_f16_plan(int T, int K, int N, int g, int M, int B, int path, int* info,
                       int n_info) {
  return linear_plan_impl(T, K, N, g, M, B, path, true, false, info, n_info);
}

int aq_linear_a16_plan(int T, int K, int N, int g, int M, int B, int path, int* info,
                       int n_info) {
  return linear_plan_impl(T, K, N, g, M, B, path, true, true, info, n_info);
}

int aq_linear(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
              const void* scale, const void* bias, void* y, int out_dtype, int T, int K, int N,
              int g, int M, int B, void* workspace, size_t workspace_bytes, int path,
              void* stream) {
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d: F16 or F32 (int8: aq_linear_q8; codes: aq_linear_ex)", out_dtype);
  return linear_impl(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, T, K, N,
                     g, M, B, workspace, workspace_bytes, path, stream);
}

int aq_linear_q8(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
                 const void* scale, const void* bias, int8_t* yq, float s_out, int T, int K,
                 int N, int g, int M, int B, void* workspace, size_t workspace_bytes, int path,
                 void* stream) {
  return linear_impl(xq, s_x, codes_packed, codebooks, scale, bias, yq, AQ_DTYPE_I8, s_out, T, K,
                     N, g, M, B, workspace, workspace_bytes, path, stream);
}

// aq_linear from fp16 activations: the workspace starts with the quantized activations
// (T*K*2 bytes, 1 KB-aligned: int8 codes, or on the dense paths the codes as fp16 values),
// then what the layer needs.
static size_t f16_act_bytes(int T, int K) { return align_up(static_cast<size_t>(T) * K * 2, 1024); }

int aq_linear_f16_workspace_size(int T, int K, int N, int g, int M, int B, int path,
                                 size_t* bytes) {
  size_t rest = 0;
  const int r = linear_ws(T, K, N, g, M, B, path, kActF16, &rest);
  if (r) return r;
  *bytes = f16_act_bytes(T, K) + rest;
  return ok();
}

int aq_linear_a16_workspace_size(int T, int K, int N, int g, int M, int B, int path,
                                 size_t* bytes) {
  const int rp = resolve_a16_path(path);
  if (rp < 0) return path_error(-2, path);
  return linear_ws(T, K, N, g, M, B, rp, kActF16Codes, bytes);
}

int aq_linear_a16(const void* xh, float s_x, const void* codes_packed, const void* codebooks,
                  const void* scale, const void* bias, void* y, int out_dtype, int T, int K, int N,
                  int g, int M, int B, void* workspace, size_t workspace_bytes, int path,
                  void* stream) {
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d: F16 or F32 (int8: aq_linear_q8; codes: aq_linear_ex)", out_dtype);
  const int rp = resolve_a16_path(path);
  if (rp < 0) return path_error(-2, path);
  if (T > 0 && !xh) return set_error(AQ_ERR_NULL, "xh is NULL");
  return linear_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, T, K,
                     N, g, M, B, workspace, workspace_bytes, rp, stream, nullptr,
                     T > 0 ? xh : nullptr);
}

int aq_linear_f16(const void* x, float s_x, const void* codes_packed, const void* codebooks,
                  const void* scale, const void* bias, void* y, int out_dtype, int T, int K, int N,
                  int g, int M, int B, void* workspace, size_t workspace_bytes, int path,
                  void* stream) {
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d: F16 or F32 (int8: aq_linear_q8; codes: aq_linear_ex)", out_dtype);
  if (!(s_x > 0.0f) || s_x == __builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite and > 0");
  if (T < 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and K > 0");
  if (T == 0)  // argument checks only, as aq_linear
    return linear_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, 0,
                       K, N, g, M, B, workspace, workspace_bytes, path, stream);
  if (!x) return set_error(AQ_ERR_NULL, "x is NULL");
  if (!aligned16(x)) return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  const size_t xq_bytes = f16_act_bytes(T, K);
  if (!workspace || workspace_bytes < xq_bytes || !aligned16(workspace))
    return set_error(AQ_ERR_WORKSPACE, "workspace needs at least %zu bytes (got %zu)", xq_bytes,
                     workspace_bytes);
  int8_t* xq = static_cast<int8_t*>(workspace);
  void* rest = static_cast<uint8_t*>(workspace) + xq_bytes;
  return linear_impl(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, T, K, N,
                     g, M, B, rest, workspace_bytes - xq_bytes, path, stream, x);
}

}  // extern "C"

namespace {

int linear_ws(int T, int K, int N, int g, int M, int B, int path, ActKind act, size_t* bytes) {
  if (!bytes) return set_error(AQ_ERR_NULL, "bytes is NULL");
  int r = check_format(g, M, B);
  if (r) return r;
  if (T < 0 || N <= 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and N, K > 0");
  if (K % 16 != 0 || N % 8 != 0) return set_error(AQ_ERR_SHAPE, "need K %% 16 == 0 and N %% 8 == 0");
  const int rp = resolve_linear_path(path, T, B, N, K, M);
  if (rp < 0) return path_error(rp, path);
  if (rp == AQ_PATH_FEW_TOKENS) {
    *bytes = 0;
    return ok();
  }
  if (rp == AQ_PATH_LUT) {
    *bytes = plan_lut(T, K, N, M).ws_bytes;
    return ok();
  }
  *bytes = route_layer(rp, T, N, K, (T + aq::kBM - 1) / aq::kBM, false, M, B, act).ws;
  return ok();
}

// x16 != nullptr (aq_linear_f16): the fp16 activations, quantized into xq by this call
// (int8 codes, or on the dense paths the codes as fp16 values: the region holds T*K*2 bytes).
// xh != nullptr (aq_linear_a16): activations already held as fp16 values; path is a
// resolved dense path and xq is unused.
int linear_impl(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
                const void* scale, const void* bias, void* y, int out_dtype, float s_out, int T,
                int K, int N, int g, int M, int B, void* workspace, size_t workspace_bytes,
                int path, void* stream, const void* x16, const void* xh) {
  int r = check_format(g, M, B);
  if (r) return r;
  if (T < 0 || N <= 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and N, K > 0");
  if (K % 16 != 0 || N % 8 != 0) return set_error(AQ_ERR_SHAPE, "need K %% 16 == 0 and N %% 8 == 0");
  r = check_output(out_dtype, s_out, N);
  if (r) return r;
  if (!(s_x == s_x) || s_x == __builtin_inff() || s_x == -__builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite");
  const int rp = resolve_linear_path(path, T, B, N, K, M);
  if (rp < 0) return path_error(rp, path);
  if (T == 0) return ok();
  const void* act = xh ? xh : static_cast<const void*>(xq);
  if (!act || !codes_packed || !codebooks || !scale || !y) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(act) || !aligned16(codes_packed) || !aligned16(codebooks) || !aligned16(scale) ||
      !aligned16(y) || (bias && !aligned16(bias)))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  if (x16 && (rp == AQ_PATH_FEW_TOKENS || rp == AQ_PATH_LUT)) {
    ProfScope ps(kProfQuant, static_cast<cudaStream_t>(stream));
    const cudaError_t e = aq::launch_quant_act(x16, const_cast<int8_t*>(xq),
                                               static_cast<int64_t>(T) * K, s_x,
                                               static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_status(e, "quantizer launch");
  }
  if (rp == AQ_PATH_FEW_TOKENS) {
    aq::SkinnyParams sp{};
    sp.xq = xq;
    sp.codes = codes_packed;
    sp.books = codebooks;
    sp.scale = static_cast<const __half*>(scale);
    sp.bias = static_cast<const __half*>(bias);
    sp.y = y;
    sp.out_f32 = out_dtype == AQ_DTYPE_F32;
    sp.out_q8 = out_codes(out_dtype);
    sp.s_x = s_x;
    sp.s_out = s_out;
    sp.T = T;
    sp.K = K;
    sp.N = N;
    sp.M = M;
    sp.B = B;
    sp.sms = sm_count();
    ProfScope ps(kProfLutGather, static_cast<cudaStream_t>(stream));
    return cuda_status(aq::launch_skinny(sp, static_cast<cudaStream_t>(stream)),
                       "few-token launch");
  }
  if (rp == AQ_PATH_LUT) {
    const LutPlan lp = plan_lut(T, K, N, M);
    if (!workspace || workspace_bytes < lp.ws_bytes || !aligned16(workspace))
      return set_error(AQ_ERR_WORKSPACE, "workspace needs %zu bytes (got %zu)", lp.ws_bytes,
                       workspace_bytes);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    aq::LutParams lpar{};
    lpar.xq = xq;
    lpar.packed = static_cast<const uint8_t*>(codes_packed);
    lpar.books = static_cast<const __half*>(codebooks);
    lpar.partial = static_cast<float*>(workspace);
    lpar.T = T;
    lpar.K = K;
    lpar.N = N;
    lpar.M = M;
    lpar.vec = lp.vec;
    lpar.Tp = lp.Tp;
    lpar.J = lp.J;
    lpar.G = K / 8;
    lpar.chunks = lp.chunks;
    lpar.rows_per_cta = lp.rows_per_cta;
    lpar.ctas = std::min(std::min(lp.ctas, sm_count()), aq::kLutrMaxCtas);
    if (lp.vec == 2)
      lutr_partition(static_cast<int64_t>(lp.chunks) * ((N + 31) / 32), (N + 31) / 32, lpar.ctas,
                     lpar.unit_bounds);
    cudaError_t e;
    {
      ProfScope ps(kProfLutGather, st);
      e = aq::launch_lut(lpar, st);
    }
    if (e != cudaSuccess) return cuda_status(e, "LUT launch");
    aq::GemmParams rpar{};
    rpar.T = T;
    rpar.N = N;
    rpar.s_x = s_x;
    rpar.scale = static_cast<const __half*>(scale);
    rpar.bias = static_cast<const __half*>(bias);
    rpar.y = y;
    rpar.out_f32 = out_dtype == AQ_DTYPE_F32;
    rpar.out_q8 = out_codes(out_dtype);
    rpar.s_out = s_out;
    rpar.partial = lpar.partial;
    {
      ProfScope ps(kProfSplitK, st);
      e = lp.vec == 2 ? aq::launch_lut_reduce(rpar, lp.chunks, st)
                      : aq::launch_splitk_reduce(rpar, lp.chunks, st);
    }
    if (e != cudaSuccess) return cuda_status(e, "LUT reduce launch");
    return ok();
  }
  // fp16 activations (given as codes, or quantized by this call) on the dense paths may run
  // the shared-memory A form (route_layer)
  const Route rt = route_layer(rp, T, N, K, (T + aq::kBM - 1) / aq::kBM,
                               out_dtype == AQ_DTYPE_F32, M, B,
                               xh ? kActF16Codes : (x16 ? kActF16 : kActInt8));
  const bool a16 = rt.pl.a16 != 0;
  r = check_workspace(workspace, workspace_bytes, rt.ws);
  if (r) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* Wdec = nullptr;
  float* partial = nullptr;
  ws_pointers(rt, workspace, N, K, &Wdec, &partial);
  CUtensorMap mapA;
  r = a16 ? encode_linear_a16(&mapA, act, T, K) : encode_linear_a(&mapA, xq, T, K);
  if (r) return r;
  aq::GemmParams p{};
  p.T = T;
  p.N = N;
  p.K = K;
  p.conv = 0;
  p.s_x = s_x;
  p.scale = static_cast<const __half*>(scale);
  p.bias = static_cast<const __half*>(bias);
  p.y = y;
  p.out_f32 = out_dtype == AQ_DTYPE_F32;
  p.out_q8 = out_codes(out_dtype);
  p.s_out = s_out;
  return run_gemm(mapA, p, rt.pl, codes_packed, codebooks, M, B, Wdec, partial, st, false, x16,
                  const_cast<int8_t*>(xq), rt.predecoded);
}

}  // namespace

extern "C" {

int aq_conv2d_workspace_size(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride,
                             int pad, int g, int M, int B, int path, size_t* bytes) {
  return conv_ws(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, kActInt8, bytes);
}

namespace {
int conv_plan_impl(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                   int g, int M, int B, int path, ActKind act, int* info, int n_info) {
  int r = check_format(g, M, B, true);
  if (r) return r;
  r = check_conv_args(Nb, H, W, Cin, Cout, kh, kw, stride, pad);
  if (r) return r;
  ConvGeom cg;
  r = conv_geometry(Nb, H, W, kh, kw, stride, pad, &cg);
  if (r) return r;
  const int rp = act == kActF16Codes ? resolve_a16_path(path) : resolve_conv_path(path, cg.m_tiles, g);
  if (rp < 0) return path_error(rp, path);
  const Route rt = route_layer(rp, Nb * cg.Ho * cg.Wo, Cout, kh * kw * Cin, cg.m_tiles, false, M,
                               B, act);
  return fill_plan_info(rp, &rt.pl, info, n_info);
}
}  // namespace

int aq_conv2d_plan(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                   int g, int M, int B, int path, int* info, int n_info) {
  return conv_plan_impl(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, kActInt8, info,
                        n_info);
}

int aq_conv2d_f16_plan(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride,
                       int pad, int g, int M, int B, int path, int* info, int n_info) {
  return conv_plan_impl(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, kActF16, info,
                        n_info);
}

int aq_conv2d_f16_workspace_size(int Nb, int H, int W, int Cin, int Cout, int kh, int kw,
                                 int stride, int pad, int g, int M, int B, int path,
                                 size_t* bytes) {
  size_t rest = 0;
  const int r = conv_ws(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, kActF16, &rest);
  if (r) return r;
  *bytes = f16_act_bytes(Nb * H * W, Cin) + rest;
  return ok();
}

int aq_conv2d_nhwc_f16(const void* x, float s_x, const void* codes_packed, const void* codebooks,
                       const void* scale, const void* bias, void* y, int out_dtype, int Nb, int H,
                       int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g,
                       int M, int B, void* workspace, size_t workspace_bytes, int path,
                       void* stream) {
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED,
                     "out_dtype %d: F16 or F32 (int8: aq_conv2d_nhwc_q8; codes: aq_conv2d_nhwc_ex)",
                     out_dtype);
  if (!(s_x > 0.0f) || s_x == __builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite and > 0");
  if (Nb < 0 || H <= 0 || W <= 0 || Cin <= 0)
    return set_error(AQ_ERR_SHAPE, "conv sizes must be positive (Nb >= 0)");
  if (Nb == 0)  // argument checks only, as aq_conv2d_nhwc
    return conv_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, 0, H,
                     W, Cin, Cout, kh, kw, stride, pad, g, M, B, workspace, workspace_bytes, path,
                     stream);
  if (!x) return set_error(AQ_ERR_NULL, "x is NULL");
  if (!aligned16(x)) return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  const size_t xq_bytes = f16_act_bytes(Nb * H * W, Cin);
  if (!workspace || workspace_bytes < xq_bytes || !aligned16(workspace))
    return set_error(AQ_ERR_WORKSPACE, "workspace needs at least %zu bytes (got %zu)", xq_bytes,
                     workspace_bytes);
  int8_t* xq = static_cast<int8_t*>(workspace);
  void* rest = static_cast<uint8_t*>(workspace) + xq_bytes;
  return conv_impl(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, Nb, H, W,
                   Cin, Cout, kh, kw, stride, pad, g, M, B, rest, workspace_bytes - xq_bytes, path,
                   stream, x);
}

int aq_conv2d_nhwc(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
                   const void* scale, const void* bias, void* y, int out_dtype, int Nb, int H,
                   int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g, int M,
                   int B, void* workspace, size_t workspace_bytes, int path, void* stream) {
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED,
                     "out_dtype %d: F16 or F32 (int8: aq_conv2d_nhwc_q8; codes: aq_conv2d_nhwc_ex)",
                     out_dtype);
  return conv_impl(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, 0.0f, Nb, H, W,
                   Cin, Cout, kh, kw, stride, pad, g, M, B, workspace, workspace_bytes, path,
                   stream);
}

int aq_conv2d_nhwc_q8(const int8_t* xq, float s_x, const void* codes_packed,
                      const void* codebooks, const void* scale, const void* bias, int8_t* yq,
                      float s_out, int Nb, int H, int W, int Cin, int Cout, int kh, int kw,
                      int stride, int pad, int g, int M, int B, void* workspace,
                      size_t workspace_bytes, int path, void* stream) {
  return conv_impl(xq, s_x, codes_packed, codebooks, scale, bias, yq, AQ_DTYPE_I8, s_out, Nb, H,
                   W, Cin, Cout, kh, kw, stride, pad, g, M, B, workspace, workspace_bytes, path,
                   stream);
}

// ---- layer calls with the activation and output kinds as arguments: int8 codes or the codes
// held as fp16 values in; fp16, fp32, int8 codes or fp16 codes out (so a chain of layers can
// hand each layer its activations in the form its tensor-core plan reads).
namespace {
int act_kind(int act_dtype, ActKind* act) {
  if (act_dtype == AQ_DTYPE_I8) {
    *act = kActInt8;
    return AQ_OK;
  }
  if (act_dtype == AQ_DTYPE_F16_CODES) {
    *act = kActF16Codes;
    return AQ_OK;
  }
  return set_error(AQ_ERR_UNSUPPORTED, "act_dtype %d: AQ_DTYPE_I8 or AQ_DTYPE_F16_CODES",
                   act_dtype);
}
}  // namespace

int aq_linear_ex_workspace_size(int act_dtype, int T, int K, int N, int g, int M, int B, int path,
                                size_t* bytes) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  if (act == kActInt8) return linear_ws(T, K, N, g, M, B, path, kActInt8, bytes);
  const int rp = resolve_a16_path(path);
  if (rp < 0) return path_error(-2, path);
  return linear_ws(T, K, N, g, M, B, rp, kActF16Codes, bytes);
}

int aq_linear_ex_plan(int act_dtype, int T, int K, int N, int g, int M, int B, int path, int* info,
                      int n_info) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  return linear_plan_impl(T, K, N, g, M, B, path, act == kActF16Codes, act == kActF16Codes, info,
                          n_info);
}

int aq_linear_ex(const void* act_in, int act_dtype, float s_x, const void* codes_packed,
                 const void* codebooks, const void* scale, const void* bias, void* y,
                 int out_dtype, float s_out, int T, int K, int N, int g, int M, int B,
                 void* workspace, size_t workspace_bytes, int path, void* stream) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  if (act == kActInt8)
    return linear_impl(static_cast<const int8_t*>(act_in), s_x, codes_packed, codebooks, scale,
                       bias, y, out_dtype, s_out, T, K, N, g, M, B, workspace, workspace_bytes,
                       path, stream);
  const int rp = resolve_a16_path(path);
  if (rp < 0) return path_error(-2, path);
  if (T > 0 && !act_in) return set_error(AQ_ERR_NULL, "activations are NULL");
  return linear_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, s_out, T,
                     K, N, g, M, B, workspace, workspace_bytes, rp, stream, nullptr,
                     T > 0 ? act_in : nullptr);
}

int aq_conv2d_ex_workspace_size(int act_dtype, int Nb, int H, int W, int Cin, int Cout, int kh,
                                int kw, int stride, int pad, int g, int M, int B, int path,
                                size_t* bytes) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  return conv_ws(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, act, bytes);
}

int aq_conv2d_ex_plan(int act_dtype, int Nb, int H, int W, int Cin, int Cout, int kh, int kw,
                      int stride, int pad, int g, int M, int B, int path, int* info, int n_info) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  return conv_plan_impl(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, path, act, info,
                        n_info);
}

int aq_conv2d_nhwc_ex(const void* act_in, int act_dtype, float s_x, const void* codes_packed,
                      const void* codebooks, const void* scale, const void* bias, void* y,
                      int out_dtype, float s_out, int Nb, int H, int W, int Cin, int Cout, int kh,
                      int kw, int stride, int pad, int g, int M, int B, void* workspace,
                      size_t workspace_bytes, int path, void* stream) {
  ActKind act;
  int r = act_kind(act_dtype, &act);
  if (r) return r;
  if (act == kActInt8)
    return conv_impl(static_cast<const int8_t*>(act_in), s_x, codes_packed, codebooks, scale, bias,
                     y, out_dtype, s_out, Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B,
                     workspace, workspace_bytes, path, stream);
  if (Nb > 0 && !act_in) return set_error(AQ_ERR_NULL, "activations are NULL");
  if (Nb == 0)  // argument checks only (the int8 form's, on a dense path)
    return conv_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, s_out, 0,
                     H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, workspace, workspace_bytes,
                     path == AQ_PATH_AUTO ? AQ_PATH_DENSE : path, stream);
  return conv_impl(nullptr, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, s_out, Nb, H,
                   W, Cin, Cout, kh, kw, stride, pad, g, M, B, workspace, workspace_bytes, path,
                   stream, nullptr, act_in);
}

}  // extern "C"

namespace {

// x16 != nullptr (aq_conv2d_nhwc_f16): the fp16 NHWC activations, quantized into xq by this
// call -- as the codes' fp16 values (the region holds Nb*H*W*Cin*2 bytes) when the
// shared-memory A form runs (route_layer), else as int8 codes.
// xh != nullptr (aq_conv2d_nhwc_ex with AQ_DTYPE_F16_CODES): the codes already held as fp16
// values; the path resolves to a dense one and xq is unused.
int conv_impl(const int8_t* xq, float s_x, const void* codes_packed, const void* codebooks,
              const void* scale, const void* bias, void* y, int out_dtype, float s_out, int Nb,
              int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g, int M,
              int B, void* workspace, size_t workspace_bytes, int path, void* stream,
              const void* x16, const void* xh) {
  int r = check_format(g, M, B, true);
  if (r) return r;
  r = check_conv_args(Nb, H, W, Cin, Cout, kh, kw, stride, pad);
  if (r) return r;
  r = check_output(out_dtype, s_out, Cout);
  if (r) return r;
  if (!(s_x == s_x) || s_x == __builtin_inff() || s_x == -__builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite");
  ConvGeom cg;
  r = conv_geometry(Nb, H, W, kh, kw, stride, pad, &cg);
  if (r) return r;
  const int rp = xh ? resolve_a16_path(path) : resolve_conv_path(path, cg.m_tiles, g);
  if (rp < 0) return path_error(rp, path);
  if (Nb == 0) return ok();
  const void* act = xh ? xh : static_cast<const void*>(xq);
  if (!act || !codes_packed || !codebooks || !scale || !y) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(act) || !aligned16(codes_packed) || !aligned16(codebooks) || !aligned16(scale) ||
      !aligned16(y) || (bias && !aligned16(bias)))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  const int K = kh * kw * Cin;
  const int T = Nb * cg.Ho * cg.Wo;
  // fp16 activations (given as codes, or quantized by this call) may run the shared-memory A
  // form (route_layer)
  const Route rt = route_layer(rp, T, Cout, K, cg.m_tiles, out_dtype == AQ_DTYPE_F32, M, B,
                               xh ? kActF16Codes : (x16 ? kActF16 : kActInt8));
  const bool a16 = rt.pl.a16 != 0;
  r = check_workspace(workspace, workspace_bytes, rt.ws);
  if (r) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* Wdec = nullptr;
  float* partial = nullptr;
  ws_pointers(rt, workspace, Cout, K, &Wdec, &partial);
  CUtensorMap mapA;
  {
    // element size 1 (int8 codes, 64-byte swizzle) or 2 (fp16 codes, 128-byte swizzle: the
    // 64-channel box row is one 128-byte swizzle span, the layout of the weight boxes)
    const cuuint64_t es_bytes = a16 ? 2 : 1;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(Cin), static_cast<cuuint64_t>(W),
                          static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(Nb)};
    cuuint64_t strides[3] = {es_bytes * Cin, es_bytes * W * Cin, es_bytes * H * W * Cin};
    // stride s: the box spans s*bw x s*bh input pixels and delivers every s-th one
    cuuint32_t box[4] = {static_cast<cuuint32_t>(aq::kBK), static_cast<cuuint32_t>(stride * cg.bw),
                         static_cast<cuuint32_t>(stride * cg.bh), static_cast<cuuint32_t>(cg.bn)};
    cuuint32_t es[4] = {1, static_cast<cuuint32_t>(stride), static_cast<cuuint32_t>(stride), 1};
    r = encode(&mapA, a16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 4,
               act, dims, strides, box,
               a16 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B, es);
    if (r) return r;
  }
  aq::GemmParams p{};
  p.T = T;
  p.N = Cout;
  p.K = K;
  p.conv = 1;
  p.cin_blocks = Cin / aq::kBK;
  p.pad = pad;
  p.stride = stride;
  p.tiles_per_img = cg.tiles_per_img;
  p.rows_per_tile = cg.rows_per_tile;
  p.imgs_per_tile = cg.imgs_per_tile;
  p.s_x = s_x;
  p.scale = static_cast<const __half*>(scale);
  p.bias = static_cast<const __half*>(bias);
  p.y = y;
  p.out_f32 = out_dtype == AQ_DTYPE_F32;
  p.out_q8 = out_codes(out_dtype);
  p.s_out = s_out;
  return run_gemm(mapA, p, rt.pl, codes_packed, codebooks, M, B, Wdec, partial, st,
                  g == kKaqGroup, x16, const_cast<int8_t*>(xq), rt.predecoded,
                  static_cast<int64_t>(Nb) * H * W * Cin);
}

int conv_ws(int Nb, int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int g,
            int M, int B, int path, ActKind act, size_t* bytes) {
  if (!bytes) return set_error(AQ_ERR_NULL, "bytes is NULL");
  int r = check_format(g, M, B, true);
  if (r) return r;
  r = check_conv_args(Nb, H, W, Cin, Cout, kh, kw, stride, pad);
  if (r) return r;
  ConvGeom cg;
  r = conv_geometry(Nb, H, W, kh, kw, stride, pad, &cg);
  if (r) return r;
  const int rp = act == kActF16Codes ? resolve_a16_path(path) : resolve_conv_path(path, cg.m_tiles, g);
  if (rp < 0) return path_error(rp, path);
  const int K = kh * kw * Cin;
  const int T = Nb * cg.Ho * cg.Wo;
  *bytes = route_layer(rp, T, Cout, K, cg.m_tiles, false, M, B, act).ws;
  return ok();
}

}  // namespace

// ---- input gradient (dL/dX through the AQ layer)
namespace {
// Workspace: [Wt fp16 K x N (+ the GEMM's split-K partials): the fp16-activation GEMM's
// predecoded workspace for the (T, K_red = N, N_out = K) contraction][ones fp16 K].
struct GradRoute {
  Route rt;
  size_t ones_off, bytes;
};

GradRoute route_input_grad(int T, int K, int N, bool f32_out, int M, int B) {
  GradRoute gr;
  gr.rt = route_gemm(AQ_PATH_PREDECODED, T, K, N, (T + aq::kBM - 1) / aq::kBM, f32_out, M, B, true);
  gr.ones_off = align_up(gr.rt.ws, 1024);
  gr.bytes = gr.ones_off + align_up(static_cast<size_t>(K) * 2, 1024);
  return gr;
}

int check_grad_shapes(int T, int K, int N, int g, int M, int B) {
  int r = check_format(g, M, B);
  if (r) return r;
  if (T < 0 || N <= 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and N, K > 0");
  if (K % 16 != 0 || N % 16 != 0)
    return set_error(AQ_ERR_SHAPE, "input gradient needs K %% 16 == 0 and N %% 16 == 0");
  return AQ_OK;
}
}  // namespace

extern "C" int aq_linear_input_grad_workspace_size(int T, int K, int N, int g, int M, int B,
                                                   size_t* bytes) {
  if (!bytes) return set_error(AQ_ERR_NULL, "bytes is NULL");
  const int r = check_grad_shapes(T, K, N, g, M, B);
  if (r) return r;
  // the same plan (and workspace) for fp16 and fp32 output
  *bytes = route_input_grad(T, K, N, false, M, B).bytes;
  return ok();
}

extern "C" int aq_linear_input_grad(const void* dy, float alpha, const void* codes_packed,
                                    const void* codebooks, const void* scale, void* dx,
                                    int out_dtype, int T, int K, int N, int g, int M, int B,
                                    void* workspace, size_t workspace_bytes, void* stream) {
  int r = check_grad_shapes(T, K, N, g, M, B);
  if (r) return r;
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d", out_dtype);
  if (!(alpha == alpha) || alpha == __builtin_inff() || alpha == -__builtin_inff())
    return set_error(AQ_ERR_SHAPE, "alpha must be finite");
  if (T == 0) return ok();
  if (!dy || !codes_packed || !codebooks || !scale || !dx) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(dy) || !aligned16(codes_packed) || !aligned16(codebooks) || !aligned16(scale) ||
      !aligned16(dx))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  // the plan for this output type: the workspace query's plan, with fp32 staging if needed
  const GradRoute gq = route_input_grad(T, K, N, false, M, B);
  const GradRoute gr = route_input_grad(T, K, N, out_dtype == AQ_DTYPE_F32, M, B);
  if (gr.bytes > gq.bytes)
    return set_error(AQ_ERR_WORKSPACE, "internal: plan for fp32 output needs more workspace");
  r = check_workspace(workspace, workspace_bytes, gq.bytes);
  if (r) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  void* Wt = nullptr;
  float* partial = nullptr;
  ws_pointers(gr.rt, workspace, K, N, &Wt, &partial);
  __half* ones = reinterpret_cast<__half*>(static_cast<uint8_t*>(workspace) + gq.ones_off);
  cudaError_t e;
  {
    ProfScope ps(kProfDecode, st);
    e = aq::launch_decode_t(codes_packed, codebooks, static_cast<const __half*>(scale),
                            static_cast<__half*>(Wt), ones, N, K, M, B, st);
  }
  if (e != cudaSuccess) return cuda_status(e, "transposed decode launch");
  // dX = alpha * dY Wt^T: the fp16-activation GEMM over (T, K_red = N, N_out = K), its
  // epilogue scale alpha * ones[k], no bias
  CUtensorMap mapA;
  r = encode_linear_a16(&mapA, dy, T, N);
  if (r) return r;
  aq::GemmParams p{};
  p.T = T;
  p.N = K;
  p.K = N;
  p.conv = 0;
  p.s_x = alpha;
  p.scale = ones;
  p.bias = nullptr;
  p.y = dx;
  p.out_f32 = out_dtype == AQ_DTYPE_F32;
  return run_gemm(mapA, p, gr.rt.pl, codes_packed, codebooks, M, B, Wt, partial, st, false,
                  nullptr, nullptr, true);
}

// Device address of g_noalloc_scratch on the current device (the host-side symbol is only
// a stand-in, never a device address), looked up once per device and context: a context
// re-created on that device (cudaDeviceReset) gets the array at a new address.
namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_dev_ptr[kMaxDevices] = {};
CUcontext g_noalloc_ctx[kMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
CtxGetCurrentFn ctx_get_current_fn() {
  static CtxGetCurrentFn fn = []() -> CtxGetCurrentFn {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    return reinterpret_cast<CtxGetCurrentFn>(p);
  }();
  return fn;
}

int noalloc_scratch_ptr(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_status(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(AQ_ERR_CUDA, "device ordinal %d out of range", dev);
  CUcontext ctx = nullptr;
  CtxGetCurrentFn get_ctx = ctx_get_current_fn();
  if (get_ctx == nullptr || get_ctx(&ctx) != CUDA_SUCCESS) ctx = nullptr;
  std::lock_guard<std::mutex> g(g_noalloc_mu);
  if (g_noalloc_dev_ptr[dev] == nullptr || ctx == nullptr || g_noalloc_ctx[dev] != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_status(e, "cudaGetSymbolAddress(no-alloc scratch)");
    if (p == nullptr || !aligned16(p)) return set_error(AQ_ERR_CUDA, "no-alloc scratch address invalid");
    g_noalloc_dev_ptr[dev] = p;
    g_noalloc_ctx[dev] = ctx;
  }
  *out = g_noalloc_dev_ptr[dev];
  return AQ_OK;
}
}  // namespace

extern "C" int aq_linear_noalloc(const int8_t* xq, float s_x, const void* codes_packed,
                                 const void* codebooks, const void* scale, const void* bias,
                                 void* y, int out_dtype, int T, int K, int N, int g, int M, int B,
                                 void* stream) {
  int r = check_format(g, M, B);
  if (r) return r;
  if (T < 0 || N <= 0 || K <= 0) return set_error(AQ_ERR_SHAPE, "need T >= 0 and N, K > 0");
  if (K % 16 != 0 || N % 8 != 0) return set_error(AQ_ERR_SHAPE, "need K %% 16 == 0 and N %% 8 == 0");
  const size_t need = static_cast<size_t>(N) * static_cast<size_t>(K) * 2;
  if (need > AQ_NOALLOC_SCRATCH_BYTES)
    return set_error(AQ_ERR_WORKSPACE,
                     "aq_linear_noalloc: N*K*2 = %zu bytes exceeds the fixed scratch of %u bytes",
                     need, (unsigned)AQ_NOALLOC_SCRATCH_BYTES);
  if (out_dtype != AQ_DTYPE_F16 && out_dtype != AQ_DTYPE_F32)
    return set_error(AQ_ERR_UNSUPPORTED, "out_dtype %d", out_dtype);
  if (!(s_x == s_x) || s_x == __builtin_inff() || s_x == -__builtin_inff())
    return set_error(AQ_ERR_SHAPE, "s_x must be finite");
  if (T == 0) return ok();
  if (!xq || !codes_packed || !codebooks || !scale || !y) return set_error(AQ_ERR_NULL, "NULL argument");
  if (!aligned16(xq) || !aligned16(codes_packed) || !aligned16(codebooks) || !aligned16(scale) ||
      !aligned16(y) || (bias && !aligned16(bias)))
    return set_error(AQ_ERR_ALIGN, "buffers must be 16-byte aligned");
  void* Wdec = nullptr;
  r = noalloc_scratch_ptr(&Wdec);
  if (r) return r;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  // no K split: the scratch holds only the decoded weights
  const Plan pl = plan_gemm(T, N, K, (T + aq::kBM - 1) / aq::kBM, false, out_dtype == AQ_DTYPE_F32);
  CUtensorMap mapA;
  r = encode_linear_a(&mapA, xq, T, K);
  if (r) return r;
  aq::GemmParams p{};
  p.T = T;
  p.N = N;
  p.K = K;
  p.conv = 0;
  p.s_x = s_x;
  p.scale = static_cast<const __half*>(scale);
  p.bias = static_cast<const __half*>(bias);
  p.y = y;
  p.out_f32 = out_dtype == AQ_DTYPE_F32;
  return run_gemm(mapA, p, pl, codes_packed, codebooks, M, B, Wdec, nullptr, st);
}
