// C ABI of the BD-LRU scan library (declared in include/blr.h): host-side
// validation, the tiling plan, workspace clearing and kernel launches. The
// library allocates nothing and never synchronises except in
// blr_workspace_status().
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <mutex>

#include <cudaTypedefs.h>

#include "blr.h"
#include "blr_chain.cuh"
#include "blr_chain_bwd.cuh"
#include "blr_merge.cuh"
#include "blr_seq.cuh"

namespace {

using blr::Plan;

thread_local char g_last_error[512] = "";

blr_status fail(blr_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
  return s;
}

blr_status cuda_check(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return BLR_OK;
  return fail(BLR_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

// Shared checks of the problem description; fills `plan` when B, L, D > 0.
blr_status check_desc(const blr_desc* d, Plan* plan, bool* empty_bd) {
  if (d == nullptr) return fail(BLR_ERR_INVALID_ARG, "desc is NULL");
  if (d->B < 0 || d->L < 0 || d->D < 0)
    return fail(BLR_ERR_INVALID_ARG, "negative size B=%lld L=%lld D=%lld", (long long)d->B,
                (long long)d->L, (long long)d->D);
  if (d->io != BLR_F32 && d->io != BLR_BF16)
    return fail(BLR_ERR_INVALID_ARG, "unknown io dtype %d", (int)d->io);
  if (!(d->c > 0.0f) || !isfinite(d->c))
    return fail(BLR_ERR_INVALID_ARG, "c must be finite and > 0");
  if (d->D % 8 != 0) return fail(BLR_ERR_UNSUPPORTED, "D=%lld is not a multiple of 8", (long long)d->D);
  *empty_bd = (d->B == 0 || d->D == 0);
  if (*empty_bd || d->L == 0) return BLR_OK;
  // Element offsets (b L + t) 2D + d must fit in int64; tile numbers in int32.
  if (d->B > (int64_t)1 << 40 || d->L > (int64_t)1 << 40 || d->D > (int64_t)1 << 24 ||
      (double)d->B * (double)d->L * (double)d->D > 1e18)
    return fail(BLR_ERR_UNSUPPORTED, "problem too large");
  // TMA coordinates are 32-bit and tensor-map strides below 2^40 bytes.
  if (d->B >= ((int64_t)1 << 31) || d->L >= ((int64_t)1 << 31) ||
      (double)d->L * (double)d->D * 8.0 >= (double)((int64_t)1 << 40))
    return fail(BLR_ERR_UNSUPPORTED, "problem too large for the tiled loads");
  blr::make_plan(d->B, d->L, d->D, (int)d->io, d->c, plan);
  if (plan->n_tiles_f >= ((int64_t)1 << 30) || plan->n_tiles_b >= ((int64_t)1 << 30))
    return fail(BLR_ERR_UNSUPPORTED, "too many tiles (%lld)", (long long)plan->n_tiles_b);
  if (plan->nseg > 0 && plan->n_tc * plan->n_chain >= ((int64_t)1 << 31))
    return fail(BLR_ERR_UNSUPPORTED, "too many chained tiles");
  if (plan->seq && plan->n_chain >= ((int64_t)1 << 31))
    return fail(BLR_ERR_UNSUPPORTED, "too many chains (%lld)", (long long)plan->n_chain);
  return BLR_OK;
}

blr_status need(const void* p, const char* name, size_t align) {
  if (p == nullptr) return fail(BLR_ERR_INVALID_ARG, "%s is NULL", name);
  if (!aligned(p, align)) return fail(BLR_ERR_INVALID_ARG, "%s is not %zu-byte aligned", name, align);
  return BLR_OK;
}

blr_status optional(const void* p, const char* name, size_t align) {
  if (p != nullptr && !aligned(p, align))
    return fail(BLR_ERR_INVALID_ARG, "%s is not %zu-byte aligned", name, align);
  return BLR_OK;
}

#define BLR_TRY(expr)                  \
  do {                                 \
    blr_status s_ = (expr);            \
    if (s_ != BLR_OK) return s_;       \
  } while (0)

blr_status check_ws(const Plan& plan, const void* ws, size_t ws_bytes) {
  BLR_TRY(need(ws, "ws", 16));
  if (ws_bytes < plan.bytes)
    return fail(BLR_ERR_INVALID_ARG, "ws_bytes=%zu < required %zu", ws_bytes, plan.bytes);
  return BLR_OK;
}

// Persistent grid: as many blocks as fit on the device at once, at most one
// per tile. The per-device block count of each kernel (and its shared-memory
// attribute) is set up once and cached: host time per call stays small.
struct GridCacheEntry {
  int dev;
  const void* fn;
  int threads;
  size_t smem;
  int blocks;  // blocks per SM x SMs
};
std::mutex g_grid_mutex;
GridCacheEntry g_grid_cache[64];
int g_grid_count = 0;

template <typename K>
blr_status persistent_grid(K kernel, int threads, size_t smem, int64_t n_tiles, unsigned* grid) {
  int dev = 0;
  BLR_TRY(cuda_check(cudaGetDevice(&dev), "cudaGetDevice"));
  const void* fn = reinterpret_cast<const void*>(kernel);
  int blocks = 0;
  {
    std::lock_guard<std::mutex> lock(g_grid_mutex);
    for (int i = 0; i < g_grid_count; ++i) {
      const GridCacheEntry& e = g_grid_cache[i];
      if (e.dev == dev && e.fn == fn && e.threads == threads && e.smem == smem) blocks = e.blocks;
    }
    if (blocks == 0) {
      int sms = 0, per_sm = 0;
      BLR_TRY(cuda_check(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem),
                         "set dynamic shared memory size"));
      BLR_TRY(cuda_check(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev),
                         "query SM count"));
      BLR_TRY(cuda_check(
          cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem),
          "query occupancy"));
      blocks = sms * (per_sm > 0 ? per_sm : 1);
      if (g_grid_count < 64) g_grid_cache[g_grid_count++] = {dev, fn, threads, smem, blocks};
    }
  }
  int64_t g = blocks;
  if (g > n_tiles) g = n_tiles;
  *grid = (unsigned)(g > 0 ? g : 1);
  return BLR_OK;
}

// cuTensorMapEncodeTiled, through the runtime's driver entry point (the
// library links only the CUDA runtime).
blr_status tensor_map_encoder(PFN_cuTensorMapEncodeTiled_v12000* out) {
  static std::mutex m;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::lock_guard<std::mutex> lock(m);
  if (fn == nullptr) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    const cudaError_t e =
        cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || ptr == nullptr)
      return fail(BLR_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
    fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  *out = fn;
  return BLR_OK;
}

// A 3-D tensor map over `cols` columns of a row-major (B, L, row_elems)
// tensor (row_elems = cols unless given), seen as (cols, L, B); boxes of
// `box_cols` columns x `rows` steps x 1 batch row. Loads read elements
// outside the view as zero; stores skip them.
blr_status make_tensor_map(CUtensorMap* map, const void* base, int io, int64_t cols, int64_t L,
                           int64_t B, int64_t rows, uint32_t box_cols = 32, int64_t row_elems = 0) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = nullptr;
  BLR_TRY(tensor_map_encoder(&enc));
  const cuuint64_t es = (io == BLR_F32) ? 4 : 2;
  if (row_elems <= 0) row_elems = cols;
  const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)L, (cuuint64_t)B};
  const cuuint64_t strides[2] = {(cuuint64_t)row_elems * es, (cuuint64_t)row_elems * es * (cuuint64_t)L};
  const cuuint32_t box[3] = {box_cols, (cuuint32_t)rows, 1u};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  const CUresult r = enc(map, io == BLR_F32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
                         3, const_cast<void*>(base), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(BLR_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return BLR_OK;
}

// Launches a scan kernel cooperatively: its blocks wait on one another, so
// all of them must be resident at once.
template <typename K, typename A>
blr_status launch_cooperative(K kernel, unsigned grid, int threads, size_t smem, cudaStream_t st,
                              const A& args, const char* what) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3((unsigned)threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cuda_check(cudaLaunchKernelEx(&cfg, kernel, args), what);
}

// ----------------------------------------------------------- serial kernels
//
// One warp per block, one block per chain. The ring's stage count is sized so
// that the blocks that share an SM (chains / SMs of them) fit its shared memory.

int sm_count() {
  static std::mutex m;
  static int counts[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  std::lock_guard<std::mutex> lock(m);
  if (counts[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    counts[dev] = n;
  }
  return counts[dev];
}

int seq_stages(int64_t n_chain, size_t stage_bytes) {
  constexpr size_t kBudget = 200u << 10;  // shared memory per SM given to the rings
  int64_t per_sm = (n_chain + sm_count() - 1) / sm_count();
  if (per_sm < 1) per_sm = 1;
  if (per_sm > 32) per_sm = 32;  // blocks per SM at most
  int64_t s = (int64_t)(kBudget / (size_t)per_sm / stage_bytes);
  if (s < 2) s = 2;
  if (s > blr::kSeqMaxStages) s = blr::kSeqMaxStages;
  return (int)s;
}

template <typename K>
blr_status allow_smem(K kernel, size_t smem) {
  if (smem <= (48u << 10)) return BLR_OK;
  return cuda_check(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                    "set dynamic shared memory size");
}

// Blocks of a serial kernel: one per chain, or per (segment, chain).
int64_t seq_blocks(const Plan& p, int mode) {
  return mode == blr::kSeqSeg ? p.n_chain * p.nseg : p.n_chain;
}

// float32 rings deep enough run the LATE form (refill after the next stage's
// arithmetic); bfloat16 always the early one.
template <typename T>
bool late_refill(int stages) {
  return sizeof(T) == 4 && stages >= blr::kSeqLateRefillStages;
}

template <typename T, class M, int VEC, int R, int RB, bool GATED, int MODE = blr::kSeqPlain>
blr_status launch_seq_fwd(blr::SeqFwdArgs& a, cudaStream_t st) {
  constexpr int NB = GATED ? 4 : 3;
  const int64_t blocks = seq_blocks(a.p, MODE);
  a.stages = seq_stages(blocks, NB * (size_t)blr::seq_box_bytes<T, VEC, R>());
  const size_t smem = blr::seq_smem_bytes<T, VEC, R>(a.stages, NB);
  auto kernel = blr::seq_fwd_kernel<T, M, VEC, R, RB, GATED, MODE, false>;
  if constexpr (sizeof(T) == 4) {
    if (late_refill<T>(a.stages)) kernel = blr::seq_fwd_kernel<T, M, VEC, R, RB, GATED, MODE, true>;
  }
  BLR_TRY(allow_smem(kernel, smem));
  kernel<<<(unsigned)blocks, 32, smem, st>>>(a);
  return cuda_check(cudaGetLastError(), "launch seq_fwd_kernel");
}

template <typename T, class M, int VEC, int R, int RB, bool GATED, int MODE = blr::kSeqPlain>
blr_status launch_seq_bwd(blr::SeqBwdArgs& a, cudaStream_t st) {
  constexpr int NB = GATED ? 5 : 4;
  const int64_t blocks = seq_blocks(a.p, MODE);
  a.stages = seq_stages(blocks, NB * (size_t)blr::seq_box_bytes<T, VEC, R>());
  const size_t smem = blr::seq_smem_bytes<T, VEC, R>(a.stages, NB);
  auto kernel = blr::seq_bwd_kernel<T, M, VEC, R, RB, GATED, MODE, false>;
  if constexpr (sizeof(T) == 4) {
    if (late_refill<T>(a.stages)) kernel = blr::seq_bwd_kernel<T, M, VEC, R, RB, GATED, MODE, true>;
  }
  BLR_TRY(allow_smem(kernel, smem));
  kernel<<<(unsigned)blocks, 32, smem, st>>>(a);
  return cuda_check(cudaGetLastError(), "launch seq_bwd_kernel");
}

// Rows per TMA box of the segment reductions (seg_len is a multiple).
constexpr int kSegReduceRows = 16;

template <typename T, class M, int VEC, bool BWD, bool GATED = false>
blr_status launch_seg_reduce(blr::SegReduceArgs& a, cudaStream_t st) {
  constexpr int R = kSegReduceRows;
  auto kernel = blr::seg_reduce_kernel<T, M, VEC, R, BWD, GATED>;
  constexpr int NB = (BWD && !GATED) ? 2 : 3;
  const int64_t blocks = a.p.n_chain * a.p.nseg;
  a.stages = seq_stages(blocks, NB * (size_t)blr::seq_box_bytes<T, VEC, R>());
  const size_t smem = blr::seq_smem_bytes<T, VEC, R>(a.stages, NB);
  BLR_TRY(allow_smem(kernel, smem));
  kernel<<<(unsigned)blocks, 32, smem, st>>>(a);
  return cuda_check(cudaGetLastError(), "launch seg_reduce_kernel");
}

// The serial kernels' views: x-shaped tensors as (D, L, B); gate_logits-shaped
// ones as two (D, L, B) views of row length 2D, at column 0 (rho) and D (iota).
blr_status seq_maps_x(CUtensorMap* m, const void* base, const Plan& plan, int rows) {
  return make_tensor_map(m, base, plan.io, plan.D, plan.L, plan.B, rows, 32u * (uint32_t)plan.sv);
}
blr_status seq_maps_gl(CUtensorMap* mr, CUtensorMap* mi, const void* base, const Plan& plan, int rows) {
  const size_t es = plan.io == BLR_F32 ? 4 : 2;
  const uint32_t cols = 32u * (uint32_t)plan.sv;
  BLR_TRY(make_tensor_map(mr, base, plan.io, plan.D, plan.L, plan.B, rows, cols, 2 * plan.D));
  return make_tensor_map(mi, static_cast<const unsigned char*>(base) + (size_t)plan.D * es, plan.io,
                         plan.D, plan.L, plan.B, rows, cols, 2 * plan.D);
}

// z given: the merge of the gated layer is fused, and h receives y = h SiLU(z).
blr_status scan_fwd_seq(const Plan& plan, const void* x, const void* gl, const float* lambda,
                        const float* h0, void* h, float* h_last, unsigned char* w, cudaStream_t st,
                        const void* z, const int32_t* lengths, bool seg = false) {
  blr::SeqFwdArgs a;
  a.lengths = lengths;
  BLR_TRY(seq_maps_x(&a.tm_x, x, plan, plan.sr));
  BLR_TRY(seq_maps_gl(&a.tm_r, &a.tm_i, gl, plan, plan.sr));
  a.write_h = h != nullptr;
  if (a.write_h) BLR_TRY(seq_maps_x(&a.tm_h, h, plan, plan.sr));
  else memset(&a.tm_h, 0, sizeof(a.tm_h));
  if (z != nullptr) BLR_TRY(seq_maps_x(&a.tm_z, z, plan, plan.sr));
  else memset(&a.tm_z, 0, sizeof(a.tm_z));
  a.p = plan;
  a.lambda = lambda;
  a.h0 = h0;
  a.h_last = h_last;
  a.ws = w;
  a.stages = 2;
  if (seg) {  // bfloat16 only (make_plan)
    constexpr int S = blr::kSeqSeg;
    if (z != nullptr) return launch_seq_fwd<__nv_bfloat16, blr::MathFast, 2, 16, 8, true, S>(a, st);
    return launch_seq_fwd<__nv_bfloat16, blr::MathFast, 2, 16, 8, false, S>(a, st);
  }
  if (z != nullptr) {
    if (plan.io == BLR_F32) {
      if (plan.sr == 32) return launch_seq_fwd<float, blr::MathPrecise, 1, 32, 16, true>(a, st);
      return launch_seq_fwd<float, blr::MathPrecise, 1, 16, 16, true>(a, st);
    }
    return launch_seq_fwd<__nv_bfloat16, blr::MathFast, 2, 16, 8, true>(a, st);
  }
  if (lengths != nullptr) {
    constexpr int V = blr::kSeqVarlen;
    if (plan.io == BLR_F32) {
      if (plan.sr == 32) return launch_seq_fwd<float, blr::MathPrecise, 1, 32, 16, false, V>(a, st);
      return launch_seq_fwd<float, blr::MathPrecise, 1, 16, 16, false, V>(a, st);
    }
    return launch_seq_fwd<__nv_bfloat16, blr::MathFast, 2, 16, 8, false, V>(a, st);
  }
  if (plan.io == BLR_F32) {
    if (plan.sr == 32) return launch_seq_fwd<float, blr::MathPrecise, 1, 32, 16, false>(a, st);
    return launch_seq_fwd<float, blr::MathPrecise, 1, 16, 16, false>(a, st);
  }
  return launch_seq_fwd<__nv_bfloat16, blr::MathFast, 2, 16, 8, false>(a, st);
}

// z and dz given: dh is dy, the gradient of y = h SiLU(z), and dz is written.
blr_status scan_bwd_seq(const Plan& plan, const void* dh, const float* dh_last, const void* x,
                        const void* gl, const float* lambda, const float* h0, void* dx, void* dgl,
                        float* dlambda, float* dh0, unsigned char* w, cudaStream_t st,
                        const void* z, void* dz, const int32_t* lengths, bool seg = false) {
  blr::SeqBwdArgs a;
  a.lengths = lengths;
  BLR_TRY(seq_maps_x(&a.tm_dh, dh, plan, plan.srb));
  BLR_TRY(seq_maps_x(&a.tm_x, x, plan, plan.srb));
  BLR_TRY(seq_maps_gl(&a.tm_r, &a.tm_i, gl, plan, plan.srb));
  BLR_TRY(seq_maps_x(&a.tm_dx, dx, plan, plan.srb));
  BLR_TRY(seq_maps_gl(&a.tm_dr, &a.tm_di, dgl, plan, plan.srb));
  const bool gated = z != nullptr;
  if (gated) {
    BLR_TRY(seq_maps_x(&a.tm_z, z, plan, plan.srb));
    BLR_TRY(seq_maps_x(&a.tm_dz, dz, plan, plan.srb));
  } else {
    memset(&a.tm_z, 0, sizeof(a.tm_z));
    memset(&a.tm_dz, 0, sizeof(a.tm_dz));
  }
  a.p = plan;
  a.dh_last = dh_last;
  a.lambda = lambda;
  a.h0 = h0;
  a.dlambda = dlambda;
  a.dh0 = dh0;
  a.ws = w;
  a.stages = 2;
  if (seg) {  // bfloat16 only (make_plan)
    constexpr int S = blr::kSeqSeg;
    if (gated) return launch_seq_bwd<__nv_bfloat16, blr::MathFast, 2, 8, 8, true, S>(a, st);
    return launch_seq_bwd<__nv_bfloat16, blr::MathFast, 2, 8, 8, false, S>(a, st);
  }
  if (gated) {
    if (plan.io == BLR_F32) return launch_seq_bwd<float, blr::MathPrecise, 1, 16, 16, true>(a, st);
    return launch_seq_bwd<__nv_bfloat16, blr::MathFast, 2, 8, 8, true>(a, st);
  }
  if (lengths != nullptr) {
    constexpr int V = blr::kSeqVarlen;
    if (plan.io == BLR_F32) return launch_seq_bwd<float, blr::MathPrecise, 1, 16, 16, false, V>(a, st);
    return launch_seq_bwd<__nv_bfloat16, blr::MathFast, 2, 8, 8, false, V>(a, st);
  }
  if (plan.io == BLR_F32) return launch_seq_bwd<float, blr::MathPrecise, 1, 16, 16, false>(a, st);
  return launch_seq_bwd<__nv_bfloat16, blr::MathFast, 2, 8, 8, false>(a, st);
}

// The segmented serial kernels (few chains, long sequences; bfloat16 I/O):
// the segment reduction, then the serial kernel over (segment, chain) blocks,
// each composing its carry from the maps.
blr_status scan_fwd_seg(const Plan& plan, const void* x, const void* gl, const float* lambda,
                        const float* h0, void* h, float* h_last, unsigned char* w,
                        cudaStream_t st, const void* z) {
  if (plan.io != BLR_BF16) return fail(BLR_ERR_UNSUPPORTED, "segmented kernels take bfloat16 I/O");
  blr::SegReduceArgs r;
  BLR_TRY(seq_maps_x(&r.tm_a, x, plan, kSegReduceRows));
  BLR_TRY(seq_maps_gl(&r.tm_r, &r.tm_i, gl, plan, kSegReduceRows));
  r.p = plan;
  r.lambda = lambda;
  r.ws = w;
  r.stages = 2;
  BLR_TRY((launch_seg_reduce<__nv_bfloat16, blr::MathFast, 2, false>(r, st)));
  return scan_fwd_seq(plan, x, gl, lambda, h0, h, h_last, w, st, z, nullptr, true);
}

blr_status scan_bwd_seg(const Plan& plan, const void* dh, const float* dh_last, const void* x,
                        const void* gl, const float* lambda, const float* h0, void* dx, void* dgl,
                        float* dlambda, float* dh0, unsigned char* w, cudaStream_t st,
                        const void* z, void* dz) {
  if (plan.io != BLR_BF16) return fail(BLR_ERR_UNSUPPORTED, "segmented kernels take bfloat16 I/O");
  blr::SegReduceArgs r;
  BLR_TRY(seq_maps_x(&r.tm_a, dh, plan, kSegReduceRows));
  BLR_TRY(seq_maps_gl(&r.tm_r, &r.tm_i, gl, plan, kSegReduceRows));
  if (z != nullptr) BLR_TRY(seq_maps_x(&r.tm_z, z, plan, kSegReduceRows));
  else memset(&r.tm_z, 0, sizeof(r.tm_z));
  r.p = plan;
  r.lambda = lambda;
  r.ws = w;
  r.stages = 2;
  if (z != nullptr)
    BLR_TRY((launch_seg_reduce<__nv_bfloat16, blr::MathFast, 2, true, true>(r, st)));
  else
    BLR_TRY((launch_seg_reduce<__nv_bfloat16, blr::MathFast, 2, true>(r, st)));
  return scan_bwd_seq(plan, dh, dh_last, x, gl, lambda, h0, dx, dgl, dlambda, dh0, w, st, z, dz,
                      nullptr, true);
}

// The chained single-pass forward (few chains, long sequences): its records
// are emptied, then one cooperative grid, one block per SM, scans every tile.
template <typename T, class M, int VEC, int RB>
blr_status launch_chain_fwd(const Plan& plan, const blr::ChainFwdArgs& a, cudaStream_t st) {
  constexpr int threads = blr::kChainThreads;
  auto k = blr::chain_fwd_kernel<T, M, VEC, RB>;
  const size_t smem = blr::ChainSmem<T, VEC>::bytes;
  unsigned grid = 1;
  BLR_TRY(persistent_grid(k, threads, smem, plan.n_tc * plan.n_chain, &grid));
  return launch_cooperative(k, grid, threads, smem, st, a, "launch chain_fwd_kernel");
}

blr_status scan_fwd_chain(const Plan& plan, const void* x, const void* gl, const float* lambda,
                          const float* h0, void* h, float* h_last, unsigned char* w,
                          cudaStream_t st) {
  if (plan.io != BLR_BF16) return fail(BLR_ERR_UNSUPPORTED, "the chained forward takes bfloat16 I/O");
  BLR_TRY(cuda_check(cudaMemsetAsync(w + plan.off_cinc, 0xff, plan.off_cend - plan.off_cinc, st),
                     "empty the chained forward's records"));
  blr::ChainFwdArgs a;
  BLR_TRY(seq_maps_x(&a.tm_x, x, plan, blr::kChainTile));
  BLR_TRY(seq_maps_gl(&a.tm_r, &a.tm_i, gl, plan, blr::kChainTile));
  a.p = plan;
  a.lambda = lambda;
  a.h0 = h0;
  a.h = h;
  a.h_last = h_last;
  a.ws = w;
  return launch_chain_fwd<__nv_bfloat16, blr::MathFast, 2, 8>(plan, a, st);
}

// The chained single-pass backward (the problems the chained forward serves,
// bfloat16): the records are emptied again (the forward's are no longer
// needed), then one cooperative grid, one block per SM.
blr_status scan_bwd_chain(const Plan& plan, const void* dh, const float* dh_last, const void* x,
                          const void* gl, const float* lambda, const float* h0, void* dx, void* dgl,
                          float* dlambda, float* dh0, unsigned char* w, cudaStream_t st) {
  if (plan.io != BLR_BF16) return fail(BLR_ERR_UNSUPPORTED, "the chained backward takes bfloat16 I/O");
  BLR_TRY(cuda_check(cudaMemsetAsync(w + plan.off_cinc, 0xff, plan.off_cend - plan.off_cinc, st),
                     "empty the chained backward's records"));
  blr::ChainBwdArgs a;
  BLR_TRY(seq_maps_x(&a.tm_dh, dh, plan, blr::kChainTile));
  BLR_TRY(seq_maps_x(&a.tm_x, x, plan, blr::kChainTile));
  BLR_TRY(seq_maps_gl(&a.tm_r, &a.tm_i, gl, plan, blr::kChainTile));
  BLR_TRY(seq_maps_x(&a.tm_dx, dx, plan, blr::kChainTile));
  BLR_TRY(seq_maps_gl(&a.tm_dr, &a.tm_di, dgl, plan, blr::kChainTile));
  a.p = plan;
  a.dh_last = dh_last;
  a.lambda = lambda;
  a.h0 = h0;
  a.dlambda = dlambda;
  a.dh0 = dh0;
  a.ws = w;
  using bf = __nv_bfloat16;
  auto k = blr::chain_bwd_kernel<bf, blr::MathFast, 2, 8>;
  const size_t smem = blr::ChainBwdSmem<bf, 2>::bytes;
  unsigned grid = 1;
  BLR_TRY(persistent_grid(k, blr::kCbThreads, smem, plan.n_tc * plan.n_chain, &grid));
  return launch_cooperative(k, grid, blr::kCbThreads, smem, st, a, "launch chain_bwd_kernel");
}

// Clears [zero, zero + zero_bytes), fills [fill, fill + fill_bytes) with the
// empty record pattern and writes k = -c softplus(Lambda).
blr_status launch_prep(unsigned char* zero, size_t zero_bytes, unsigned char* fill,
                       size_t fill_bytes, float* k, const float* lambda, int64_t D, float c,
                       cudaStream_t st) {
  const int64_t words = (int64_t)(zero_bytes / 4);
  const int64_t vec4 = (int64_t)(fill_bytes / 16);
  int64_t work = words > D ? words : D;
  if (vec4 > work) work = vec4;
  int64_t blocks = (work + 255) / 256;
  if (blocks > 2048) blocks = 2048;
  blr::prep_kernel<<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<uint32_t*>(zero), words,
                                                     reinterpret_cast<uint4*>(fill), vec4, k,
                                                     lambda, D, c);
  return cuda_check(cudaGetLastError(), "launch prep_kernel");
}

template <typename T, class M, bool VARLEN>
blr_status launch_tiled_fwd(const Plan& plan, const blr::FwdArgs& a, cudaStream_t st) {
  const int threads = (plan.nwarps + 1) * 32;  // consumer warps + the scanner warp
  auto k = blr::scan_fwd_kernel<T, M, VARLEN>;
  const size_t smem = blr::ring_bytes<T, blr::fwd_stages<T>(), 3>();
  unsigned grid = 1;
  BLR_TRY(persistent_grid(k, threads, smem, plan.n_tiles_f, &grid));
  return launch_cooperative(k, grid, threads, smem, st, a, "launch scan_fwd_kernel");
}

template <typename T, class M, bool VARLEN>
blr_status launch_tiled_bwd(const Plan& plan, const blr::BwdArgs& a, cudaStream_t st) {
  const int threads = plan.nwarps * 32;
  auto k = blr::scan_bwd_kernel<T, M, VARLEN>;
  const size_t smem = blr::ring_bytes<T, blr::bwd_stages<T>(), 4>();
  unsigned grid = 1;
  BLR_TRY(persistent_grid(k, threads, smem, plan.n_tiles_b, &grid));
  return launch_cooperative(k, grid, threads, smem, st, a, "launch scan_bwd_kernel");
}

// The tiled look-back kernels: a preparation kernel, then the scan.
blr_status scan_fwd_tiled(const Plan& plan, const blr_desc* desc, const void* x,
                          const void* gate_logits, const float* lambda, const float* h0, void* h,
                          float* h_last, unsigned char* w, cudaStream_t st,
                          const int32_t* lengths) {
  // Clear the forward header (counters, error word), empty the
  // forward records, precompute k = -c softplus(Lambda).
  BLR_TRY(launch_prep(w + plan.off_fhdr, sizeof(blr::FwdHeader), w + plan.off_fpre,
                      plan.off_frec_end - plan.off_fpre, reinterpret_cast<float*>(w + plan.off_k),
                      lambda, desc->D, desc->c, st));
  blr::FwdArgs a;
  a.lengths = lengths;
  BLR_TRY(make_tensor_map(&a.tm_x, x, desc->io, desc->D, desc->L, desc->B, plan.tsteps));
  BLR_TRY(make_tensor_map(&a.tm_gl, gate_logits, desc->io, 2 * desc->D, desc->L, desc->B, plan.tsteps));
  a.p = plan;
  a.h0 = h0;
  a.h = h;
  a.h_last = h_last;
  a.ws = w;
  if (desc->io == BLR_F32) {
    if (lengths != nullptr) return launch_tiled_fwd<float, blr::MathPrecise, true>(plan, a, st);
    return launch_tiled_fwd<float, blr::MathPrecise, false>(plan, a, st);
  }
  if (lengths != nullptr) return launch_tiled_fwd<__nv_bfloat16, blr::MathFast, true>(plan, a, st);
  return launch_tiled_fwd<__nv_bfloat16, blr::MathFast, false>(plan, a, st);
}

// dh may be the dx buffer itself: every element of dh is read (into shared
// memory, with its tile) before its tile writes dx.
blr_status scan_bwd_tiled(const Plan& plan, const blr_desc* desc, const void* dh,
                          const float* dh_last, const void* x, const void* gate_logits,
                          const float* lambda, const float* h0, void* dx, void* dgate_logits,
                          float* dlambda, float* dh0, unsigned char* w, cudaStream_t st,
                          const int32_t* lengths) {
  // Clear the backward header and the dLambda partial sums, empty the backward
  // records (the forward's records stay: they hold the carries).
  BLR_TRY(launch_prep(w + plan.off_bhdr, plan.off_k - plan.off_bhdr, w + plan.off_bagg,
                      plan.bytes - plan.off_bagg, reinterpret_cast<float*>(w + plan.off_k), lambda,
                      desc->D, desc->c, st));
  blr::BwdArgs a;
  a.lengths = lengths;
  BLR_TRY(make_tensor_map(&a.tm_dh, dh, desc->io, desc->D, desc->L, desc->B, plan.tsteps));
  BLR_TRY(make_tensor_map(&a.tm_x, x, desc->io, desc->D, desc->L, desc->B, plan.tsteps));
  BLR_TRY(make_tensor_map(&a.tm_gl, gate_logits, desc->io, 2 * desc->D, desc->L, desc->B, plan.tsteps));
  a.p = plan;
  a.dh_last = dh_last;
  a.lambda = lambda;
  a.h0 = h0;
  a.dx = dx;
  a.dgl = dgate_logits;
  a.dlambda = dlambda;
  a.dh0 = dh0;
  a.ws = w;
  if (desc->io == BLR_F32) {
    if (lengths != nullptr) return launch_tiled_bwd<float, blr::MathPrecise, true>(plan, a, st);
    return launch_tiled_bwd<float, blr::MathPrecise, false>(plan, a, st);
  }
  if (lengths != nullptr) return launch_tiled_bwd<__nv_bfloat16, blr::MathFast, true>(plan, a, st);
  return launch_tiled_bwd<__nv_bfloat16, blr::MathFast, false>(plan, a, st);
}

// Grid of the elementwise merge kernels: 16-byte vectors, 256 threads a block,
// at most 8 blocks per SM (grid-stride beyond).
unsigned merge_grid(int64_t n_vec) {
  int64_t blocks = (n_vec + 255) / 256;
  const int64_t cap = (int64_t)sm_count() * 8;
  if (blocks > cap) blocks = cap;
  return (unsigned)(blocks > 0 ? blocks : 1);
}

blr_status launch_merge_fwd(int io, void* y, const void* z, int64_t n, cudaStream_t st) {
  if (io == BLR_F32) {
    const int64_t nv = n / 4;
    blr::merge_fwd_kernel<float><<<merge_grid(nv), 256, 0, st>>>(static_cast<float*>(y),
                                                                 static_cast<const float*>(z), nv);
  } else {
    const int64_t nv = n / 8;
    blr::merge_fwd_kernel<__nv_bfloat16><<<merge_grid(nv), 256, 0, st>>>(
        static_cast<__nv_bfloat16*>(y), static_cast<const __nv_bfloat16*>(z), nv);
  }
  return cuda_check(cudaGetLastError(), "launch merge_fwd_kernel");
}

blr_status launch_merge_bwd(int io, const void* dy, const void* z, void* dh, void* hz, int64_t n,
                            cudaStream_t st) {
  if (io == BLR_F32) {
    const int64_t nv = n / 4;
    blr::merge_bwd_kernel<float><<<merge_grid(nv), 256, 0, st>>>(
        static_cast<const float*>(dy), static_cast<const float*>(z), static_cast<float*>(dh),
        static_cast<float*>(hz), nv);
  } else {
    const int64_t nv = n / 8;
    using bf = __nv_bfloat16;
    blr::merge_bwd_kernel<bf><<<merge_grid(nv), 256, 0, st>>>(
        static_cast<const bf*>(dy), static_cast<const bf*>(z), static_cast<bf*>(dh),
        static_cast<bf*>(hz), nv);
  }
  return cuda_check(cudaGetLastError(), "launch merge_bwd_kernel");
}

// The library's static device scratch (defined with blr_scan_fwd_noalloc):
// its size, and its address on the current device after checking that the
// problem's workspace fits (BLR_ERR_UNSUPPORTED, nothing enqueued, if not).
constexpr size_t kLibraryScratchBytes = (size_t)128 << 20;  // 128 MiB
blr_status library_scratch(const Plan& plan, const char* who, void** out);

// blr_scan_fwd (z == NULL) and blr_scan_fwd_gated (z given; h is then y).
blr_status scan_fwd_entry(const blr_desc* desc, const void* x, const void* gate_logits,
                          const float* lambda, const float* h0, const void* z, void* h,
                          float* h_last, void* ws, size_t ws_bytes, blr_stream_t stream,
                          bool gated, const int32_t* lengths = nullptr, bool varlen = false) {
  Plan plan;
  bool empty = false;
  BLR_TRY(check_desc(desc, &plan, &empty));
  if (empty) return BLR_OK;
  BLR_TRY(need(lambda, "lambda", 16));
  BLR_TRY(optional(h0, "h0", 4));
  BLR_TRY(optional(h_last, "h_last", 4));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const size_t state_bytes = sizeof(float) * (size_t)desc->B * (size_t)desc->D;
  if (desc->L == 0) {  // empty sequence: the state is unchanged
    if (h_last == nullptr) return BLR_OK;
    if (h0 != nullptr)
      return cuda_check(cudaMemcpyAsync(h_last, h0, state_bytes, cudaMemcpyDeviceToDevice, st),
                        "copy h0 to h_last");
    return cuda_check(cudaMemsetAsync(h_last, 0, state_bytes, st), "clear h_last");
  }
  BLR_TRY(need(x, "x", 16));
  BLR_TRY(need(gate_logits, "gate_logits", 16));
  BLR_TRY(optional(h, gated ? "y" : "h", 16));
  if (gated) BLR_TRY(need(z, "z", 16));
  if (varlen) BLR_TRY(need(lengths, "lengths", 4));
  BLR_TRY(check_ws(plan, ws, ws_bytes));

  unsigned char* w = static_cast<unsigned char*>(ws);
  if (plan.seq)  // serial kernels (the merge fused): no preparation
    return scan_fwd_seq(plan, x, gate_logits, lambda, h0, h, h_last, w, st,
                        h != nullptr ? z : nullptr, lengths);
  // Few long chains: the chained single-pass forward, or with the gated
  // layer's merge the segmented serial kernels (the merge fused); rows with
  // lengths on these problems run the tiled kernels. Either forward leaves the
  // kept states the segmented backward starts from.
  if (plan.nseg > 0 && lengths == nullptr) {
    if (z == nullptr || h == nullptr)
      return scan_fwd_chain(plan, x, gate_logits, lambda, h0, h, h_last, w, st);
    return scan_fwd_seg(plan, x, gate_logits, lambda, h0, h, h_last, w, st, z);
  }
  BLR_TRY(scan_fwd_tiled(plan, desc, x, gate_logits, lambda, h0, h, h_last, w, st, lengths));
  if (z == nullptr || h == nullptr) return BLR_OK;
  return launch_merge_fwd(desc->io, h, z, desc->B * desc->L * desc->D, st);
}

// blr_scan_bwd (z == NULL; dh is the gradient of h) and blr_scan_bwd_gated
// (z and dz given; dh is the gradient dy of y = h SiLU(z)).
blr_status scan_bwd_entry(const blr_desc* desc, const void* dh, const float* dh_last, const void* x,
                          const void* gate_logits, const float* lambda, const float* h0,
                          const void* z, void* dx, void* dgate_logits, void* dz, float* dlambda,
                          float* dh0, void* ws, size_t ws_bytes, blr_stream_t stream, bool gated,
                          const int32_t* lengths = nullptr, bool varlen = false) {
  Plan plan;
  bool empty = false;
  BLR_TRY(check_desc(desc, &plan, &empty));
  if (empty) return BLR_OK;
  BLR_TRY(need(lambda, "lambda", 16));
  BLR_TRY(need(dlambda, "dlambda", 4));
  BLR_TRY(optional(h0, "h0", 4));
  BLR_TRY(optional(dh_last, "dh_last", 4));
  BLR_TRY(optional(dh0, "dh0", 4));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (desc->L == 0) {  // empty sequence: dh0 = dh_last, no dependence on Lambda
    const size_t state_bytes = sizeof(float) * (size_t)desc->B * (size_t)desc->D;
    BLR_TRY(cuda_check(cudaMemsetAsync(dlambda, 0, sizeof(float) * (size_t)desc->D, st),
                       "clear dlambda"));
    if (dh0 == nullptr) return BLR_OK;
    if (dh_last != nullptr)
      return cuda_check(cudaMemcpyAsync(dh0, dh_last, state_bytes, cudaMemcpyDeviceToDevice, st),
                        "copy dh_last to dh0");
    return cuda_check(cudaMemsetAsync(dh0, 0, state_bytes, st), "clear dh0");
  }
  BLR_TRY(need(dh, gated ? "dy" : "dh", 16));
  if (gated) {
    BLR_TRY(need(z, "z", 16));
    BLR_TRY(need(dz, "dz", 16));
  }
  if (varlen) BLR_TRY(need(lengths, "lengths", 4));
  BLR_TRY(need(x, "x", 16));
  BLR_TRY(need(gate_logits, "gate_logits", 16));
  BLR_TRY(need(dx, "dx", 16));
  BLR_TRY(need(dgate_logits, "dgate_logits", 16));
  if (ws == nullptr) {
    // No workspace: recompute the forward's carries (a forward without h) in
    // the library's scratch, then run the backward from them.
    void* scratch = nullptr;
    BLR_TRY(library_scratch(plan, "a backward without a workspace", &scratch));
    BLR_TRY(scan_fwd_entry(desc, x, gate_logits, lambda, h0, nullptr, nullptr, nullptr, scratch,
                           kLibraryScratchBytes, stream, false, lengths, varlen));
    ws = scratch;
    ws_bytes = kLibraryScratchBytes;
  }
  BLR_TRY(check_ws(plan, ws, ws_bytes));

  unsigned char* w = static_cast<unsigned char*>(ws);
  if (plan.seq)  // the forward cleared the counters and partial sums
    return scan_bwd_seq(plan, dh, dh_last, x, gate_logits, lambda, h0, dx, dgate_logits, dlambda,
                        dh0, w, st, z, dz, lengths);
  if (plan.nseg > 0 && lengths == nullptr) {
    if (z == nullptr)
      return scan_bwd_chain(plan, dh, dh_last, x, gate_logits, lambda, h0, dx, dgate_logits,
                            dlambda, dh0, w, st);
    return scan_bwd_seg(plan, dh, dh_last, x, gate_logits, lambda, h0, dx, dgate_logits, dlambda,
                        dh0, w, st, z, dz);
  }
  if (z == nullptr)
    return scan_bwd_tiled(plan, desc, dh, dh_last, x, gate_logits, lambda, h0, dx, dgate_logits,
                          dlambda, dh0, w, st, lengths);
  // Gated, tiled: h recomputed into dz (a forward of the same problem, which
  // also rewrites the same carries), then dh = dy SiLU(z) into dx and
  // dz = dy h SiLU'(z), then the scan's backward from dh in dx.
  BLR_TRY(scan_fwd_tiled(plan, desc, x, gate_logits, lambda, h0, dz, nullptr, w, st, nullptr));
  BLR_TRY(launch_merge_bwd(desc->io, dh, z, dx, dz, desc->B * desc->L * desc->D, st));
  return scan_bwd_tiled(plan, desc, dx, dh_last, x, gate_logits, lambda, h0, dx, dgate_logits,
                        dlambda, dh0, w, st, nullptr);
}

}  // namespace

extern "C" {

size_t blr_workspace_bytes(const blr_desc* desc) {
  Plan plan;
  bool empty = false;
  if (check_desc(desc, &plan, &empty) != BLR_OK || empty || desc->L == 0) return 0;
  return plan.bytes;
}

int blr_scan_family(const blr_desc* desc, int with_lengths) {
  Plan plan;
  bool empty = false;
  if (check_desc(desc, &plan, &empty) != BLR_OK || empty || desc->L == 0) return BLR_FAMILY_NONE;
  if (plan.seq) return BLR_FAMILY_SERIAL;
  if (plan.nseg > 0 && !with_lengths) return BLR_FAMILY_SEGMENTED;
  return BLR_FAMILY_TILED;
}

blr_status blr_scan_fwd(const blr_desc* desc, const void* x, const void* gate_logits,
                        const float* lambda, const float* h0, void* h, float* h_last, void* ws,
                        size_t ws_bytes, blr_stream_t stream) {
  return scan_fwd_entry(desc, x, gate_logits, lambda, h0, nullptr, h, h_last, ws, ws_bytes, stream,
                        false);
}

blr_status blr_scan_fwd_gated(const blr_desc* desc, const void* x, const void* gate_logits,
                              const float* lambda, const float* h0, const void* z, void* y,
                              float* h_last, void* ws, size_t ws_bytes, blr_stream_t stream) {
  return scan_fwd_entry(desc, x, gate_logits, lambda, h0, z, y, h_last, ws, ws_bytes, stream, true);
}

blr_status blr_scan_fwd_varlen(const blr_desc* desc, const int32_t* lengths, const void* x,
                               const void* gate_logits, const float* lambda, const float* h0,
                               void* h, float* h_last, void* ws, size_t ws_bytes,
                               blr_stream_t stream) {
  return scan_fwd_entry(desc, x, gate_logits, lambda, h0, nullptr, h, h_last, ws, ws_bytes, stream,
                        false, lengths, true);
}

blr_status blr_scan_bwd_varlen(const blr_desc* desc, const int32_t* lengths, const void* dh,
                               const float* dh_last, const void* x, const void* gate_logits,
                               const float* lambda, const float* h0, void* dx, void* dgate_logits,
                               float* dlambda, float* dh0, void* ws, size_t ws_bytes,
                               blr_stream_t stream) {
  return scan_bwd_entry(desc, dh, dh_last, x, gate_logits, lambda, h0, nullptr, dx, dgate_logits,
                        nullptr, dlambda, dh0, ws, ws_bytes, stream, false, lengths, true);
}

blr_status blr_scan_bwd(const blr_desc* desc, const void* dh, const float* dh_last, const void* x,
                        const void* gate_logits, const float* lambda, const float* h0, void* dx,
                        void* dgate_logits, float* dlambda, float* dh0, void* ws, size_t ws_bytes,
                        blr_stream_t stream) {
  return scan_bwd_entry(desc, dh, dh_last, x, gate_logits, lambda, h0, nullptr, dx, dgate_logits,
                        nullptr, dlambda, dh0, ws, ws_bytes, stream, false);
}

blr_status blr_scan_bwd_gated(const blr_desc* desc, const void* dy, const float* dh_last,
                              const void* x, const void* gate_logits, const float* lambda,
                              const float* h0, const void* z, void* dx, void* dgate_logits,
                              void* dz, float* dlambda, float* dh0, void* ws, size_t ws_bytes,
                              blr_stream_t stream) {
  return scan_bwd_entry(desc, dy, dh_last, x, gate_logits, lambda, h0, z, dx, dgate_logits, dz,
                        dlambda, dh0, ws, ws_bytes, stream, true);
}

blr_status blr_step(int64_t B, int64_t D, blr_dtype io, float c, const float* h_prev,
                    const void* x_t, const void* gate_logits_t, const float* lambda, float* h_t,
                    blr_stream_t stream) {
  if (B < 0 || D < 0) return fail(BLR_ERR_INVALID_ARG, "negative size B=%lld D=%lld", (long long)B, (long long)D);
  if (io != BLR_F32 && io != BLR_BF16) return fail(BLR_ERR_INVALID_ARG, "unknown io dtype %d", (int)io);
  if (!(c > 0.0f) || !isfinite(c)) return fail(BLR_ERR_INVALID_ARG, "c must be finite and > 0");
  if (D % 8 != 0) return fail(BLR_ERR_UNSUPPORTED, "D=%lld is not a multiple of 8", (long long)D);
  if (B == 0 || D == 0) return BLR_OK;
  if (D > (int64_t)1 << 24 || B > (int64_t)1 << 40) return fail(BLR_ERR_UNSUPPORTED, "problem too large");
  BLR_TRY(need(h_prev, "h_prev", 16));
  BLR_TRY(need(x_t, "x_t", 16));
  BLR_TRY(need(gate_logits_t, "gate_logits_t", 16));
  BLR_TRY(need(lambda, "lambda", 16));
  BLR_TRY(need(h_t, "h_t", 16));
  // f32: two rows of 4 channels a thread per step of its walk; bf16: one row of 8
  const int rows = (io == BLR_F32) ? 2 : 1;
  const int vec = (io == BLR_F32) ? 4 : 8;
  const int64_t nvec = D / vec;
  const int bx = (int)(nvec < 64 ? nvec : 64);
  const int by = 256 / bx;
  const int64_t n_vgroups = (nvec + bx - 1) / bx;
  // a persistent grid: as many row groups as fill the GPU, at most one per block row of work
  const int64_t need_rg = (B + (int64_t)by * rows - 1) / ((int64_t)by * rows);
  int64_t n_rg = ((int64_t)sm_count() * blr::kStepBlocksPerSm + n_vgroups - 1) / n_vgroups;
  if (n_rg > need_rg) n_rg = need_rg;
  if (n_rg < 1) n_rg = 1;
  if (n_vgroups * n_rg >= ((int64_t)1 << 31)) return fail(BLR_ERR_UNSUPPORTED, "grid too large");
  blr::StepArgs a{B, D, c, n_vgroups, h_prev, x_t, gate_logits_t, lambda, h_t};
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid((unsigned)(n_vgroups * n_rg)), block((unsigned)bx, (unsigned)by);
  if (io == BLR_F32)
    blr::step_kernel<float, 4, blr::MathPrecise, 2><<<grid, block, 0, st>>>(a);
  else
    blr::step_kernel<__nv_bfloat16, 8, blr::MathFast, 1><<<grid, block, 0, st>>>(a);
  return cuda_check(cudaGetLastError(), "launch step_kernel");
}

blr_status blr_steps(int64_t B, int64_t K, int64_t D, blr_dtype io, blr_dtype state, float c,
                     const void* h_prev, const void* x, const void* gate_logits,
                     const float* lambda, void* h_out, void* h_seq, blr_stream_t stream) {
  if (B < 0 || K < 0 || D < 0)
    return fail(BLR_ERR_INVALID_ARG, "negative size B=%lld K=%lld D=%lld", (long long)B, (long long)K,
                (long long)D);
  if (io != BLR_F32 && io != BLR_BF16) return fail(BLR_ERR_INVALID_ARG, "unknown io dtype %d", (int)io);
  if (state != BLR_F32 && state != BLR_BF16)
    return fail(BLR_ERR_INVALID_ARG, "unknown state dtype %d", (int)state);
  if (!(c > 0.0f) || !isfinite(c)) return fail(BLR_ERR_INVALID_ARG, "c must be finite and > 0");
  if (D % 8 != 0) return fail(BLR_ERR_UNSUPPORTED, "D=%lld is not a multiple of 8", (long long)D);
  if (B == 0 || D == 0) return BLR_OK;
  if (D > (int64_t)1 << 24 || B > (int64_t)1 << 40 || K > (int64_t)1 << 40 ||
      (double)B * (double)K * (double)D > 1e18)
    return fail(BLR_ERR_UNSUPPORTED, "problem too large");
  BLR_TRY(need(h_prev, "h_prev", 16));
  BLR_TRY(need(h_out, "h_out", 16));
  BLR_TRY(need(lambda, "lambda", 16));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (K == 0) {  // no step: the state is unchanged
    if (h_out == h_prev) return BLR_OK;
    const size_t bytes = (size_t)B * (size_t)D * (state == BLR_F32 ? 4 : 2);
    return cuda_check(cudaMemcpyAsync(h_out, h_prev, bytes, cudaMemcpyDeviceToDevice, st),
                      "copy h_prev to h_out");
  }
  BLR_TRY(need(x, "x", 16));
  BLR_TRY(need(gate_logits, "gate_logits", 16));
  BLR_TRY(optional(h_seq, "h_seq", 16));
  const int vec = io == BLR_F32 ? 4 : 8;
  const int64_t threads = B * (D / vec);
  const int64_t blocks = (threads + 255) / 256;
  if (blocks >= ((int64_t)1 << 31)) return fail(BLR_ERR_UNSUPPORTED, "grid too large");
  blr::StepsArgs a{B, K, D, c, h_prev, x, gate_logits, lambda, h_out, h_seq};
  using bf = __nv_bfloat16;
  if (io == BLR_F32) {
    if (state == BLR_F32)
      blr::steps_kernel<float, float, 4, blr::MathPrecise><<<(unsigned)blocks, 256, 0, st>>>(a);
    else
      blr::steps_kernel<float, bf, 4, blr::MathPrecise><<<(unsigned)blocks, 256, 0, st>>>(a);
  } else {
    if (state == BLR_F32)
      blr::steps_kernel<bf, float, 8, blr::MathFast><<<(unsigned)blocks, 256, 0, st>>>(a);
    else
      blr::steps_kernel<bf, bf, 8, blr::MathFast><<<(unsigned)blocks, 256, 0, st>>>(a);
  }
  return cuda_check(cudaGetLastError(), "launch steps_kernel");
}

blr_status blr_workspace_status(const blr_desc* desc, const void* ws, size_t ws_bytes,
                                blr_stream_t stream) {
  Plan plan;
  bool empty = false;
  BLR_TRY(check_desc(desc, &plan, &empty));
  if (empty || desc->L == 0) return BLR_OK;
  if (ws == nullptr) {  // the scratch of a backward called without a workspace
    void* scratch = nullptr;
    BLR_TRY(library_scratch(plan, "blr_workspace_status without a workspace", &scratch));
    ws = scratch;
    ws_bytes = kLibraryScratchBytes;
  }
  BLR_TRY(check_ws(plan, ws, ws_bytes));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint32_t err = 0;
  const unsigned char* w = static_cast<const unsigned char*>(ws);
  BLR_TRY(cuda_check(cudaMemcpyAsync(&err, w + plan.off_fhdr + offsetof(blr::FwdHeader, err),
                                     sizeof(err), cudaMemcpyDeviceToHost, st),
                     "read workspace error word"));
  BLR_TRY(cuda_check(cudaStreamSynchronize(st), "synchronize stream"));
  if (err & blr::kErrTimeout) return BLR_ERR_TIMEOUT;
  if (err & blr::kErrWorkspace) return BLR_ERR_WORKSPACE;
  return BLR_OK;
}

blr_status blr_selftest_wait_timeout(const blr_desc* desc, void* ws, size_t ws_bytes,
                                     uint64_t timeout_ns, blr_stream_t stream) {
  Plan plan;
  bool empty = false;
  BLR_TRY(check_desc(desc, &plan, &empty));
  if (empty || desc->L == 0) return fail(BLR_ERR_INVALID_ARG, "the self-test needs a non-empty problem");
  BLR_TRY(check_ws(plan, ws, ws_bytes));
  if (timeout_ns > blr::kWaitTimeoutNs) return fail(BLR_ERR_INVALID_ARG, "timeout_ns above 1e9");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned char* w = static_cast<unsigned char*>(ws);
  uint32_t* flag = reinterpret_cast<uint32_t*>(w + plan.off_bhdr + offsetof(blr::BwdHeader, selftest_flag));
  uint32_t* err = reinterpret_cast<uint32_t*>(w + plan.off_fhdr + offsetof(blr::FwdHeader, err));
  BLR_TRY(cuda_check(cudaMemsetAsync(flag, 0, sizeof(uint32_t), st), "clear self-test flag"));
  blr::selftest_wait_kernel<<<1, 32, 0, st>>>(flag, err, timeout_ns);
  return cuda_check(cudaGetLastError(), "launch selftest_wait_kernel");
}

const char* blr_status_string(blr_status status) {
  switch (status) {
    case BLR_OK: return "BLR_OK";
    case BLR_ERR_INVALID_ARG: return "BLR_ERR_INVALID_ARG: invalid argument";
    case BLR_ERR_UNSUPPORTED: return "BLR_ERR_UNSUPPORTED: unsupported problem";
    case BLR_ERR_CUDA: return "BLR_ERR_CUDA: CUDA error";
    case BLR_ERR_TIMEOUT: return "BLR_ERR_TIMEOUT: a bounded inter-block wait expired";
    case BLR_ERR_WORKSPACE: return "BLR_ERR_WORKSPACE: workspace holds no matching forward carries";
  }
  return "unknown blr_status";
}

const char* blr_last_error_string(void) { return g_last_error; }

}  // extern "C"

// ----------------------------------------------------------------------------
// Scans without a caller workspace (blr_scan_fwd_noalloc, and the backward
// entry points given ws == NULL).
//
// Some callers cannot allocate device memory at the point where they run the
// scan: code inside CUDA stream capture that may not add allocations, plugins
// whose host framework owns every device allocation, or real-time serving
// loops that forbid allocator calls. For them the scan can run on a scratch
// array that lives in the library itself: a file-scope device array of
// kLibraryScratchBytes, present on every GPU that loads this library until
// the process exits. The host never dereferences the array's name (in host
// code it is only a stand-in for the device symbol); the device address comes
// from cudaGetSymbolAddress, looked up once per device and context.

static __device__ __align__(256) unsigned char g_noalloc_scratch[kLibraryScratchBytes];

namespace {

constexpr int kMaxDevices = 64;

std::mutex g_scratch_mutex;
void* g_scratch_ptr[kMaxDevices] = {};
CUcontext g_scratch_ctx[kMaxDevices] = {};

// The calling thread's current CUDA context (NULL if none), through the
// runtime's driver entry point (the library links only the CUDA runtime).
CUcontext current_context() {
  static PFN_cuCtxGetCurrent_v4000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 4000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(ptr);
  });
  CUcontext ctx = nullptr;
  if (fn == nullptr || fn(&ctx) != CUDA_SUCCESS) return nullptr;
  return ctx;
}

// Device address of the scratch array on the current device, set up on the
// first call on each device and again whenever the device's context has
// changed since (a reset or a re-created primary context loads the module
// anew, so an address from before would be stale).
blr_status noalloc_scratch(void** out) {
  int dev = 0;
  BLR_TRY(cuda_check(cudaGetDevice(&dev), "cudaGetDevice"));
  if (dev < 0 || dev >= kMaxDevices)
    return fail(BLR_ERR_UNSUPPORTED, "device index %d above the scratch table", dev);
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  CUcontext ctx = current_context();
  if (g_scratch_ptr[dev] == nullptr || ctx == nullptr || ctx != g_scratch_ctx[dev]) {
    void* p = nullptr;
    BLR_TRY(cuda_check(cudaGetSymbolAddress(&p, g_noalloc_scratch),
                       "cudaGetSymbolAddress of the static scratch"));
    g_scratch_ptr[dev] = p;
    g_scratch_ctx[dev] = current_context();  // current now, if it was not before the lookup
  }
  *out = g_scratch_ptr[dev];
  return BLR_OK;
}

blr_status library_scratch(const Plan& plan, const char* who, void** out) {
  if (plan.bytes > kLibraryScratchBytes)
    return fail(BLR_ERR_UNSUPPORTED,
                "%s: this problem needs %zu bytes of scratch, above the %zu-byte static scratch; "
                "pass a workspace of blr_workspace_bytes",
                who, plan.bytes, kLibraryScratchBytes);
  return noalloc_scratch(out);
}

}  // namespace

extern "C" blr_status blr_scan_fwd_noalloc(const blr_desc* desc, const void* x,
                                           const void* gate_logits, const float* lambda,
                                           const float* h0, void* h, float* h_last,
                                           blr_stream_t stream) {
  Plan plan;
  bool empty = false;
  BLR_TRY(check_desc(desc, &plan, &empty));
  if (empty || desc->L == 0)  // nothing that needs scratch: the ordinary path does it
    return blr_scan_fwd(desc, x, gate_logits, lambda, h0, h, h_last, nullptr, 0, stream);
  void* scratch = nullptr;
  BLR_TRY(library_scratch(plan, "blr_scan_fwd_noalloc", &scratch));
  return blr_scan_fwd(desc, x, gate_logits, lambda, h0, h, h_last, scratch, kLibraryScratchBytes,
                      stream);
}
