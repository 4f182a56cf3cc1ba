// BD-LRU scan kernels for sm_103a: forward scan, backward reverse scan,
// single recurrent step, and the per-call preparation kernel. The path is
// elementwise and memory-bound: no tensor cores; 16-byte (or 8-byte) accesses
// along the channels, the gate arithmetic fused into the loads, float32 state.
//
// Scan structure. Persistent thread blocks (a cooperative launch: all resident)
// process tiles (tsteps time steps x CH channels of one batch row) on a static
// schedule, time-major, so a tile only ever waits for tiles of smaller number,
// which earlier or concurrent iterations of other blocks process. For one tile:
//   1. every lane loads its kTc steps x VEC channels, computes the gates and
//      folds its chunk into one affine map h -> A h + U, serially in registers;
//   2. the kNtl lanes of a warp that share channels combine their maps with
//      warp shuffles into exclusive prefix maps and a warp map;
//   3. warp 0 combines the warp maps (shared memory) into the tile map and
//      chains the tile to the tiles before it with a decoupled look-back: one
//      lane per predecessor reads its status flag, a ballot finds the nearest
//      published prefix, and the aggregates in between are folded in;
//   4. every lane applies its prefix maps to the tile's carry and re-runs its
//      chunk from the true state, writing the outputs.
// Shared state is double-buffered by tile parity, so one barrier before and
// one after warp 0's part are the only block-wide synchronisation per tile.
#pragma once

#include <cuda.h>
#include <limits.h>

#include "blr_device.cuh"

namespace blr {

constexpr unsigned kFull = 0xffffffffu;

// The first step of row b's sequence: 0, or L - lengths[b] (lengths clamped to
// [0, L]) when the rows carry their own lengths; the steps before it are
// padding (Sec. 3.3's left padding), never read and never written.
__device__ __forceinline__ int64_t row_start(const int32_t* lengths, int64_t b, int64_t L) {
  if (lengths == nullptr) return 0;
  int64_t n = lengths[b];
  n = n < 0 ? 0 : (n > L ? L : n);
  return L - n;
}

// Inputs reach the scan kernels through TMA tensor maps over 3-D views
// (channels, time, batch) of the row-major tensors: x and dh as (D, L, B),
// gate_logits as (2D, L, B).
struct FwdArgs {
  CUtensorMap tm_x;
  CUtensorMap tm_gl;
  Plan p;
  const int32_t* lengths;  // NULL, or row b's sequence is its last lengths[b] steps
  const float* h0;
  void* h;
  float* h_last;
  unsigned char* ws;
};

struct BwdArgs {
  CUtensorMap tm_dh;
  CUtensorMap tm_x;
  CUtensorMap tm_gl;
  Plan p;
  const int32_t* lengths;  // as FwdArgs
  const float* dh_last;
  const float* lambda;
  const float* h0;
  void* dx;
  void* dgl;
  float* dlambda;
  float* dh0;
  unsigned char* ws;
};

// Shared-memory ring of the scan kernels: STAGES stages of NB boxes, each box
// kMaxTile rows x 32 channels, then one mbarrier per stage.
constexpr int kMaxTile = kMaxWarps * kWarpSteps;
template <typename T>
__host__ __device__ constexpr uint32_t box_bytes() {
  return (uint32_t)(kMaxTile * 32 * sizeof(T));
}
template <typename T, int STAGES, int NB>
__host__ __device__ constexpr size_t ring_bytes() {  // + slack to align the ring to 1 KiB
  return (size_t)STAGES * NB * box_bytes<T>() + (size_t)STAGES * sizeof(uint64_t) + 1024;
}

// The ring's base: the dynamic shared memory rounded up to 1 KiB.
__device__ __forceinline__ unsigned char* ring_base(unsigned char* dyn) {
  const uint32_t a = smem_addr(dyn);
  return dyn + (((a + 1023u) & ~1023u) - a);
}
// Stages per block, sized so that four forward (three backward) blocks fit an
// SM's shared memory.
template <typename T>
__host__ __device__ constexpr int fwd_stages() {
  return sizeof(T) == 4 ? 2 : 4;
}
template <typename T>
__host__ __device__ constexpr int bwd_stages() {
  return sizeof(T) == 4 ? 2 : 3;
}

struct StepArgs {
  int64_t B, D;
  float c;
  int64_t n_vgroups;  // blocks along the channel vectors
  const float* h_prev;
  const void* x;
  const void* gl;
  const float* lambda;
  float* h_t;
};

// ------------------------------------------------------------ preparation
//
// Clears the counters of a scan (exits, partial sums), fills its
// look-back records with the empty pattern, and writes k[d] = -c softplus(Lambda_d).

__global__ void prep_kernel(uint32_t* zero, int64_t zero_words, uint4* fill, int64_t fill_vec4,
                            float* k, const float* lambda, int64_t D, float c) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t i0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (int64_t i = i0; i < zero_words; i += stride) zero[i] = 0u;
  const uint4 empty = make_uint4(kEmpty, kEmpty, kEmpty, kEmpty);
  for (int64_t i = i0; i < fill_vec4; i += stride) fill[i] = empty;
  for (int64_t d = i0; d < D; d += stride) k[d] = decay_rate(c, lambda[d]);
}

// ------------------------------------------------------- warp-level scans
//
// Lane layout: lane = tcl * kNvl + cv. The kNtl lanes with the same cv hold
// consecutive chunks in time of the same channels.

// Turns each lane's chunk map (A, U) into the inclusive prefix map of the
// chunks up to it (A, U; the last time lane then holds the warp's map) and the
// exclusive one (ea, eu).
template <int V>
__device__ __forceinline__ void warp_prefix(float (&A)[V], float (&U)[V], int tcl,
                                            float (&ea)[V], float (&eu)[V]) {
#pragma unroll
  for (int off = 1; off < kNtl; off <<= 1) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float pa = __shfl_up_sync(kFull, A[v], off * kNvl);
      const float pu = __shfl_up_sync(kFull, U[v], off * kNvl);
      if (tcl >= off) {  // (this . earlier) = (A pa, A pu + U)
        U[v] = fmaf(A[v], pu, U[v]);
        A[v] *= pa;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    ea[v] = __shfl_up_sync(kFull, A[v], kNvl);
    eu[v] = __shfl_up_sync(kFull, U[v], kNvl);
    if (tcl == 0) {
      ea[v] = 1.0f;
      eu[v] = 0.0f;
    }
  }
}

// The same from the end of the warp's time range: (A, W) becomes the map from
// the value entering after the warp's last step to the value at this lane's
// chunk start (the first time lane then holds the warp's map), and (sa, sw)
// the map to the value entering after this lane's chunk.
template <int V>
__device__ __forceinline__ void warp_suffix(float (&A)[V], float (&W)[V], int tcl,
                                            float (&sa)[V], float (&sw)[V]) {
#pragma unroll
  for (int off = 1; off < kNtl; off <<= 1) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float na = __shfl_down_sync(kFull, A[v], off * kNvl);
      const float nw = __shfl_down_sync(kFull, W[v], off * kNvl);
      if (tcl + off < kNtl) {  // (this . later) = (A na, A nw + W)
        W[v] = fmaf(A[v], nw, W[v]);
        A[v] *= na;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    sa[v] = __shfl_down_sync(kFull, A[v], kNvl);
    sw[v] = __shfl_down_sync(kFull, W[v], kNvl);
    if (tcl == kNtl - 1) {
      sa[v] = 1.0f;
      sw[v] = 0.0f;
    }
  }
}

// ---------------------------------------------------------------- look-back
//
// Run by each lane of warp 0 for its own channel. Predecessor i (i = 0 is the
// adjacent tile in scan order) has its records at agg[i * step] and
// pre[i * step]. A window of kLookWindow predecessors is read in one round
// trip; the walk folds aggregates (nearest first) until it meets a published
// prefix. The farthest predecessor (i = nprev - 1, the first tile of the
// chain) publishes only a prefix, so the walk always ends.
// The first window's loads, issued early so that their round trip overlaps
// other work (predecessors past the first tile are not read).
struct LookWindow {
  uint32_t pr[kLookWindow];
  unsigned long long ag[kLookWindow];
};

__device__ __forceinline__ void lookback_load(const unsigned long long* agg, const uint32_t* pre,
                                              int64_t step, int64_t nprev, int64_t i,
                                              LookWindow& w) {
#pragma unroll
  for (int q = 0; q < kLookWindow; ++q) {
    w.pr[q] = kEmpty;
    w.ag[q] = ~0ull;
    if (i + q < nprev) {
      w.pr[q] = ld_record(pre + (i + q) * step);
      w.ag[q] = ld_record(agg + (i + q) * step);
    }
  }
}

// Walks the predecessors starting with the window `w` (loaded for i = 0).
__device__ __forceinline__ float lookback(const unsigned long long* agg, const uint32_t* pre,
                                          int64_t step, int64_t nprev, uint32_t* err,
                                          LookWindow& w) {
  float ea = 1.0f, eu = 0.0f;  // fold of the predecessors walked so far
  int64_t i = 0;
  for (;;) {
    int adv = kLookWindow;
    bool open = true, wait = false;
#pragma unroll
    for (int q = 0; q < kLookWindow; ++q) {
      if (open) {
        if (w.pr[q] != kEmpty) return fmaf(ea, __uint_as_float(w.pr[q]), eu);
        if (agg_empty(w.ag[q])) {  // published nothing yet: wait for it, then re-read from it
          open = false;
          wait = true;
          adv = q;
        } else {
          eu = fmaf(ea, __uint_as_float((uint32_t)(w.ag[q] >> 32)), eu);
          ea *= __uint_as_float((uint32_t)w.ag[q]);
        }
      }
    }
    if (wait && !wait_record(pre + (i + adv) * step, agg + (i + adv) * step, err, kWaitTimeoutNs))
      return eu;  // the wait expired (recorded): finish with what is known
    i += adv;
    lookback_load(agg, pre, step, nprev, i, w);
  }
}

// The whole walk, loads included.
__device__ __forceinline__ float lookback(const unsigned long long* agg, const uint32_t* pre,
                                          int64_t step, int64_t nprev, uint32_t* err) {
  LookWindow w;
  lookback_load(agg, pre, step, nprev, 0, w);
  return lookback(agg, pre, step, nprev, err, w);
}

// ------------------------------------------------------------ tile schedule
//
// Static schedule: block c processes tiles c, c + G, c + 2G, ... (G blocks,
// all resident: the scans are cooperative launches), in order. Tiles are
// numbered time-major, so a tile only waits for tiles of smaller number, and
// processing order across blocks follows tile order without any queueing.

struct TileCoord {
  int64_t tile;   // the tile's number; >= the tile count means no tile
  int64_t tt;     // time tile
  int64_t cidx;   // channel group in [0, B * groups per row)
  int64_t b;      // batch row
  int64_t dbase;  // first channel of the group
};

// Tile counts stay below 2^30 (checked on the host), so 32-bit division suffices.
__device__ __forceinline__ TileCoord decode_tile(int64_t tile, int64_t n_tiles, int64_t n_c,
                                                 int64_t n_cg, int ch, int64_t n_t, bool reverse) {
  TileCoord c;
  c.tile = tile;
  c.tt = c.cidx = c.b = c.dbase = 0;
  if (tile < n_tiles) {
    const uint32_t t32 = (uint32_t)tile, nc32 = (uint32_t)n_c, ncg32 = (uint32_t)n_cg;
    const uint32_t q = t32 / nc32;
    const uint32_t cidx = t32 - q * nc32;
    const uint32_t b = cidx / ncg32;
    c.tt = reverse ? n_t - 1 - (int64_t)q : (int64_t)q;  // the backward hands tiles out from the end
    c.cidx = cidx;
    c.b = b;
    c.dbase = (int64_t)(cidx - b * ncg32) * ch;
  }
  return c;
}

// ---------------------------------------------------------- gate arithmetic
//
// e^l - 1 for l = k r <= 0: the polynomial alone when |k| <= kPolyLimit (then
// |l| <= kPolyLimit for every r in [0, 1]), else the general form.
constexpr float kPolyLimit = 0.25f;

template <class M, bool POLY>
__device__ __forceinline__ float gate_expm1(float l) {
  if (POLY) return M::expm1_poly(l);
  return M::expm1_any(l);
}

// One lane's rows of a box in a stage: rows row0 .. row0 + kTc - 1, channels
// cv*VEC .. cv*VEC + VEC - 1 (box rows are 32 channels wide).
template <class IO>
__device__ __forceinline__ void lds_rows(const unsigned char* box, int row0, int cv,
                                         typename IO::Raw (&r)[kTc]) {
  using T = typename IO::T;
  const T* base = reinterpret_cast<const T*>(box) + row0 * 32 + cv * IO::VEC;
#pragma unroll
  for (int s = 0; s < kTc; ++s) r[s] = *reinterpret_cast<const typename IO::Raw*>(base + s * 32);
}

// Forward gates of a lane's chunk: alpha and u = sqrt(1 - alpha^2) i x per
// element; FULL when every element is inside the sequence and the channels,
// else elements outside (rows before `lo` or from `valid` on) become the
// identity map (alpha = 1, u = 0).
template <class IO, class M, bool FULL>
__device__ __forceinline__ void fwd_chunk(const float (&k)[4],
                                          const typename IO::Raw (&rx)[kTc],
                                          const typename IO::Raw (&rr)[kTc],
                                          const typename IO::Raw (&ri)[kTc], int lo, int valid,
                                          float (&al)[kTc][4], float (&u)[kTc][4]) {
  float xv[kTc][4], rv[kTc][4], iv[kTc][4];
  using G = typename GatePolicy<M>::type;
  constexpr bool HALF = G::kHalfInputs && sizeof(typename IO::T) == 2;
#pragma unroll
  for (int s = 0; s < kTc; ++s) {
    if constexpr (HALF) {
      IO::unpack_half(rx[s], xv[s]);
      IO::unpack_half(rr[s], rv[s]);
      IO::unpack_half(ri[s], iv[s]);
    } else {
      IO::unpack(rx[s], xv[s]);
      IO::unpack(rr[s], rv[s]);
      IO::unpack(ri[s], iv[s]);
    }
  }
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    if (k[v] >= -kPolyLimit) {
      const float kh = 0.5f * k[v];
#pragma unroll
      for (int s = 0; s < kTc; ++s) {
        if constexpr (HALF) {
          const float e = gate_expm1<M, true>(G::decay_log_half(rv[s][v], kh));
          al[s][v] = 1.0f + e;
          u[s][v] = M::sqrt(-e * (2.0f + e)) * G::gated_x_half(iv[s][v], xv[s][v]);
        } else {
          const float r = M::sigmoid(rv[s][v]);
          const float i = M::sigmoid(iv[s][v]);
          const float e = gate_expm1<M, true>(k[v] * r);
          al[s][v] = 1.0f + e;
          u[s][v] = M::sqrt(-e * (2.0f + e)) * i * xv[s][v];
        }
      }
    } else if constexpr (HALF) {
      const float kh = 0.5f * k[v];
#pragma unroll
      for (int s = 0; s < kTc; ++s) {
        const float e = gate_expm1<M, false>(G::decay_log_half(rv[s][v], kh));
        al[s][v] = 1.0f + e;
        u[s][v] = M::sqrt(-e * (2.0f + e)) * G::gated_x_half(iv[s][v], xv[s][v]);
      }
    } else {
#pragma unroll
      for (int s = 0; s < kTc; ++s) {
        const float r = M::sigmoid(rv[s][v]);
        const float i = M::sigmoid(iv[s][v]);
        const float e = gate_expm1<M, false>(k[v] * r);
        al[s][v] = 1.0f + e;
        u[s][v] = M::sqrt(-e * (2.0f + e)) * i * xv[s][v];
      }
    }
  }
  if (!FULL) {
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      if (s < lo || s >= valid) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          al[s][v] = 1.0f;
          u[s][v] = 0.0f;
        }
      }
    }
  }
}

// ---------------------------------------------------------------- forward scan
//
// Block = nwarps consumer warps (one time sub-tile each) + one scanner warp,
// one barrier per tile. In iteration k the consumers compute tile k's gates
// and maps (the last consumer warp to finish publishes the tile's aggregate)
// while the scanner finishes tile k-1: it walks back for the carry, publishes
// the prefix, writes every warp's starting state and refills the freed TMA
// stage. After the barrier the consumers apply tile k-1 (whose alpha and u
// they kept in registers). The scanner's round trips to L2 thus overlap the
// consumers' arithmetic.

// VARLEN: the rows carry lengths (a.lengths), whose padding the kernel masks;
// the form without keeps the registers of the plain scan.
template <typename T, class M, bool VARLEN>
__global__ void __launch_bounds__((kMaxWarps + 1) * 32, sizeof(T) == 4 ? 2 : 3)
    scan_fwd_kernel(const __grid_constant__ FwdArgs a) {
  using IO = Io<T, 4>;
  using Raw = typename IO::Raw;
  constexpr int VEC = 4;
  constexpr int CH = kNvl * VEC;
  constexpr int S = fwd_stages<T>();
  constexpr int NB = 3;  // boxes per stage: x, rho, iota
  static_assert(CH == 32, "the scanner handles one channel per lane");
  const Plan& p = a.p;
  const int nw = p.nwarps;  // consumer warps

  extern __shared__ __align__(1024) unsigned char dyn_smem[];
  unsigned char* smem = ring_base(dyn_smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * NB * box_bytes<T>());
  __shared__ float2 s_wtot[2][kMaxWarps][CH];  // each warp's map of its sub-tile
  __shared__ float s_hw[2][kMaxWarps][CH];     // each warp's starting state
  __shared__ int s_done[2];                    // consumer warps past their maps

  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  unsigned long long* agg = reinterpret_cast<unsigned long long*>(a.ws + p.off_fagg);
  uint32_t* pre = reinterpret_cast<uint32_t*>(a.ws + p.off_fpre);
  const float* kd = reinterpret_cast<const float*>(a.ws + p.off_k);
  T* h = static_cast<T*>(a.h);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool scanner = warp == nw;
  const int cv = lane % kNvl, tcl = lane / kNvl;
  const int64_t BD = p.B * p.D;
  const int row0 = warp * kWarpSteps + tcl * kTc;  // this lane's first row in a tile
  const uint32_t box_tx = (uint32_t)p.tsteps * CH * sizeof(T);

  auto tile_at = [&](int64_t i) {  // this block's i-th tile
    return decode_tile(i * gridDim.x + blockIdx.x, p.n_tiles_f, p.n_c_f, p.n_cg_f, CH, p.n_t, false);
  };
  auto issue = [&](int stage, const TileCoord& c) {  // one thread: the tile's boxes into a stage
    unsigned char* dst = smem + (size_t)stage * NB * box_bytes<T>();
    const int t = (int)(c.tt * p.tsteps), d = (int)c.dbase, bb = (int)c.b;
    mbar_arrive_expect_tx(&bars[stage], NB * box_tx);
    tma_load_3d(dst, &a.tm_x, &bars[stage], d, t, bb);
    tma_load_3d(dst + box_bytes<T>(), &a.tm_gl, &bars[stage], d, t, bb);
    tma_load_3d(dst + 2 * box_bytes<T>(), &a.tm_gl, &bars[stage], (int)p.D + d, t, bb);
  };

  // Prologue: thread 0 starts the loads of the block's first S tiles.
  if (threadIdx.x < 2) s_done[threadIdx.x] = 0;
  if (threadIdx.x == 0) {
    for (int j = 0; j < S; ++j) mbar_init(&bars[j], 1);
    fence_mbar_init();
    for (int j = 0; j < S; ++j) {
      const TileCoord c = tile_at(j);
      if (c.tile < p.n_tiles_f) issue(j, c);
    }
  }
  __syncthreads();

  // Consumer state carried from tile k-1 to its apply in iteration k.
  float pal[kTc][VEC], pu[kTc][VEC], pea[VEC], peu[VEC];
  TileCoord prev;
  prev.tile = p.n_tiles_f;  // none
  prev.tt = prev.cidx = prev.b = prev.dbase = 0;
  int prev_valid = 0, prev_lo = 0;
  float nk[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) nk[v] = 0.0f;
  {
    const TileCoord c0 = tile_at(0);
    if (!scanner && c0.tile < p.n_tiles_f && c0.dbase + cv * VEC < p.D)
      load_f32<VEC>(kd + c0.dbase + cv * VEC, nk);
  }

  for (int it = 0;; ++it) {
    const TileCoord tc = tile_at(it);
    const bool cur_ok = tc.tile < p.n_tiles_f;
    const bool prev_ok = prev.tile < p.n_tiles_f;
    if (!cur_ok && !prev_ok) break;
    const int buf = it & 1;

    if (!scanner) {
      // ---- consumers: tile it, gates and maps
      float al[kTc][VEC], u[kTc][VEC], ea[VEC], eu[VEC];
      int valid = 0, lo = 0;
      if (cur_ok) {
        const int64_t d0 = tc.dbase + cv * VEC;
        const int64_t left = (d0 < p.D) ? p.L - (tc.tt * p.tsteps + row0) : 0;
        valid = (int)(left < 0 ? 0 : (left > kTc ? kTc : left));
        if constexpr (VARLEN) {
          const int64_t head = row_start(a.lengths, tc.b, p.L) - (tc.tt * p.tsteps + row0);
          lo = (int)(head < 0 ? 0 : (head > kTc ? kTc : head));
        }
        float k[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) k[v] = nk[v];
        {
          const TileCoord c = tile_at(it + 1);
#pragma unroll
          for (int v = 0; v < VEC; ++v) nk[v] = 0.0f;
          if (c.tile < p.n_tiles_f && c.dbase + cv * VEC < p.D)
            load_f32<VEC>(kd + c.dbase + cv * VEC, nk);
        }
        const int stage = it % S;
        mbar_wait(&bars[stage], (uint32_t)(it / S) & 1u, &fh->err);
        const unsigned char* sb = smem + (size_t)stage * NB * box_bytes<T>();
        Raw rx[kTc], rr[kTc], ri[kTc];
        lds_rows<IO>(sb, row0, cv, rx);
        lds_rows<IO>(sb + box_bytes<T>(), row0, cv, rr);
        lds_rows<IO>(sb + 2 * box_bytes<T>(), row0, cv, ri);
        if (valid == kTc && lo == 0)
          fwd_chunk<IO, M, true>(k, rx, rr, ri, lo, valid, al, u);
        else
          fwd_chunk<IO, M, false>(k, rx, rr, ri, lo, valid, al, u);
        float A[VEC], U[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          A[v] = al[0][v];
          U[v] = u[0][v];
#pragma unroll
          for (int s = 1; s < kTc; ++s) {
            U[v] = fmaf(al[s][v], U[v], u[s][v]);
            A[v] *= al[s][v];
          }
        }
        warp_prefix<VEC>(A, U, tcl, ea, eu);
        if (tcl == kNtl - 1) {
#pragma unroll
          for (int v = 0; v < VEC; ++v) s_wtot[buf][warp][cv * VEC + v] = make_float2(A[v], U[v]);
        }
        // The last consumer warp to get here publishes the tile's aggregate at
        // once: successors in time may be waiting for it.
        __syncwarp();
        __threadfence_block();
        int last = 0;
        if (lane == 0) last = atomicAdd(&s_done[buf], 1) == nw - 1;
        last = __shfl_sync(kFull, last, 0);
        if (last) {
          __threadfence_block();
          const int ch = lane;
          if (tc.tt > 0 && tc.dbase + ch < p.D) {
            float pa = 1.0f, pu2 = 0.0f;
            for (int w = 0; w < nw; ++w) {
              const float2 e = s_wtot[buf][w][ch];
              pu2 = fmaf(e.x, pu2, e.y);
              pa *= e.x;
            }
            st_record(&agg[tc.tt * BD + tc.b * p.D + tc.dbase + ch], pack_agg(pa, pu2));
          }
          if (lane == 0) s_done[buf] = 0;
        }
      }
      __syncthreads();
      // ---- consumers: apply tile it-1 from the starting states the scanner wrote
      if (prev_ok && h != nullptr && prev_valid > prev_lo) {
        const int64_t d0 = prev.dbase + cv * VEC;
        const int64_t t0 = prev.tt * p.tsteps + row0;
        float hs[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) hs[v] = fmaf(pea[v], s_hw[buf ^ 1][warp][cv * VEC + v], peu[v]);
        T* ph = h + (prev.b * p.L + t0) * p.D + d0;
#pragma unroll
        for (int s = 0; s < kTc; ++s) {
          float out[VEC];
#pragma unroll
          for (int v = 0; v < VEC; ++v) {
            hs[v] = fmaf(pal[s][v], hs[v], pu[s][v]);
            out[v] = hs[v];
          }
          if (s >= prev_lo && s < prev_valid) IO::store(ph + s * p.D, out);
        }
      }
#pragma unroll
      for (int s = 0; s < kTc; ++s)
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          pal[s][v] = al[s][v];
          pu[s][v] = u[s][v];
        }
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        pea[v] = ea[v];
        peu[v] = eu[v];
      }
      prev_valid = valid;
      if constexpr (VARLEN) prev_lo = lo;
    } else {
      // ---- scanner: tile it-1's carry and warp states, and the freed stage's
      // refill. The first look-back window is requested before anything else,
      // so its round trip overlaps the rest.
      const int ch = lane;
      const bool cval = prev_ok && prev.dbase + ch < p.D;
      const int64_t rec = prev.tt * BD + prev.b * p.D + prev.dbase + ch;
      LookWindow win;
      if (cval && prev.tt > 0) lookback_load(agg + rec - BD, pre + rec - BD, -BD, prev.tt, 0, win);
      if (lane == 0 && it > 0) {  // the stage tile it-1 used is free: load tile it-1+S into it
        const TileCoord c = tile_at(it - 1 + S);
        if (c.tile < p.n_tiles_f) issue((it - 1) % S, c);
      }
      if (prev_ok) {
        float pa = 1.0f, pu2 = 0.0f;  // the tile's map
        for (int w = 0; w < nw; ++w) {
          const float2 e = s_wtot[buf ^ 1][w][ch];
          pu2 = fmaf(e.x, pu2, e.y);
          pa *= e.x;
        }
        float carry = 0.0f;
        if (cval) {
          if (prev.tt == 0) {
            if (a.h0 != nullptr) carry = a.h0[prev.b * p.D + prev.dbase + ch];
          } else {
            carry = lookback(agg + rec - BD, pre + rec - BD, -BD, prev.tt, &fh->err, win);
          }
          const float incl = fmaf(pa, carry, pu2);
          st_record(&pre[rec], __float_as_uint(incl));
          if (prev.tt == p.n_t - 1 && a.h_last != nullptr)
            a.h_last[prev.b * p.D + prev.dbase + ch] = incl;
        }
        float hw = carry;  // each warp's starting state: the carry through the warps before it
        for (int w = 0; w < nw; ++w) {
          s_hw[buf ^ 1][w][ch] = hw;
          const float2 e = s_wtot[buf ^ 1][w][ch];
          hw = fmaf(e.x, hw, e.y);
        }
      }
      __syncthreads();
    }
    prev = tc;
  }
  // The last block out marks the forward complete (for the backward's check).
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(&fh->exited, 1u) == gridDim.x - 1) {
      fh->tag = p.tag;
      __threadfence();
      fh->complete = 1u;
    }
  }
}

// ------------------------------------------------------- backward reverse scan
//
// With g_t the total derivative w.r.t. h_t and w_t = alpha_t g_t (what step t
// hands back to step t-1), g_t = dh_t + w_{t+1} and w_t = alpha_t (dh_t + w_{t+1}):
// a first-order linear scan run from the end, with the same operator as the
// forward. Per element, with l = log(alpha), q = 1 - alpha^2, n = sqrt(q):
//   dx    = g n i
//   diota = g n x i (1 - i)                   = g u (1 - i),  u = n i x
//   dl    = g alpha (h_{t-1} - alpha i x / n) = g alpha (h_{t-1} - alpha u / q)
//   drho  = dl k r (1 - r)                    (l = k r, k = -c softplus(Lambda))
//   dLambda += dl (-c r) sigmoid(Lambda)      (summed over b, t)
// h_{t-1} is rebuilt from the forward's per-tile carries, not read from h.

// Backward first pass over a lane's chunk: keeps E = expm1(l), r, i (and
// x, dh) per element and folds the chunk's maps (A, U) forwards and W
// backwards; elements outside the sequence or the channels are the identity.
template <class IO, class M, bool FULL>
__device__ __forceinline__ void bwd_chunk(const float (&k)[4], const typename IO::Raw (&rg)[kTc],
                                          const typename IO::Raw (&rx)[kTc],
                                          const typename IO::Raw (&rr)[kTc],
                                          const typename IO::Raw (&ri)[kTc], int lo, int valid,
                                          float (&gv)[kTc][4], float (&xv)[kTc][4],
                                          float (&ev)[kTc][4], float (&rv)[kTc][4],
                                          float (&iv)[kTc][4], float (&A)[4], float (&U)[4],
                                          float (&W)[4]) {
#pragma unroll
  for (int s = 0; s < kTc; ++s) {
    IO::unpack(rg[s], gv[s]);
    IO::unpack(rx[s], xv[s]);
    IO::unpack(rr[s], rv[s]);
    IO::unpack(ri[s], iv[s]);
  }
  float uu[kTc][4];
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    if (k[v] >= -kPolyLimit) {
#pragma unroll
      for (int s = 0; s < kTc; ++s) {
        const float r = M::sigmoid(rv[s][v]);
        const float i = M::sigmoid(iv[s][v]);
        const float e = gate_expm1<M, true>(k[v] * r);
        uu[s][v] = M::sqrt(-e * (2.0f + e)) * i * xv[s][v];
        rv[s][v] = r;
        iv[s][v] = i;
        ev[s][v] = e;
      }
    } else {
#pragma unroll
      for (int s = 0; s < kTc; ++s) {
        const float r = M::sigmoid(rv[s][v]);
        const float i = M::sigmoid(iv[s][v]);
        const float e = gate_expm1<M, false>(k[v] * r);
        uu[s][v] = M::sqrt(-e * (2.0f + e)) * i * xv[s][v];
        rv[s][v] = r;
        iv[s][v] = i;
        ev[s][v] = e;
      }
    }
  }
  if (!FULL) {
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      if (s < lo || s >= valid) {
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          ev[s][v] = 0.0f;
          rv[s][v] = 0.0f;
          iv[s][v] = 0.0f;
          gv[s][v] = 0.0f;
          xv[s][v] = 0.0f;
          uu[s][v] = 0.0f;
        }
      }
    }
  }
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    A[v] = 1.0f;
    U[v] = 0.0f;
    W[v] = 0.0f;
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      const float alpha = 1.0f + ev[s][v];
      U[v] = fmaf(alpha, U[v], uu[s][v]);
      A[v] *= alpha;                      // prod of alpha up to and including s
      W[v] = fmaf(A[v], gv[s][v], W[v]);  // w at the chunk start from a zero carry
    }
  }
}

template <typename T, class M, bool VARLEN>
__global__ void __launch_bounds__(kMaxWarps * 32, 3)
    scan_bwd_kernel(const __grid_constant__ BwdArgs a) {
  using IO = Io<T, 4>;
  using Raw = typename IO::Raw;
  constexpr int VEC = 4;
  constexpr int CH = kNvl * VEC;
  constexpr int S = bwd_stages<T>();
  constexpr int NB = 4;  // boxes per stage: dh, x, rho, iota
  static_assert(CH == 32, "warp 0 handles one channel per lane");
  const Plan& p = a.p;

  extern __shared__ __align__(1024) unsigned char dyn_smem[];
  unsigned char* smem = ring_base(dyn_smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)S * NB * box_bytes<T>());
  __shared__ float s_wa[2][kMaxWarps][CH];   // warp prod alpha -> warp prefix map A
  __shared__ float s_wu[2][kMaxWarps][CH];   // warp U          -> warp prefix map U
  __shared__ float s_ww[2][kMaxWarps][CH];   // warp W          -> warp suffix map W
  __shared__ float s_ws[2][kMaxWarps][CH];   //                 -> warp suffix map A
  __shared__ float s_hc[2][CH], s_wc[2][CH];
  __shared__ int s_flag;

  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(a.ws + p.off_bhdr);
  unsigned long long* agg = reinterpret_cast<unsigned long long*>(a.ws + p.off_bagg);
  uint32_t* pre = reinterpret_cast<uint32_t*>(a.ws + p.off_bpre);
  const float* fpre = reinterpret_cast<const float*>(a.ws + p.off_fpre);
  const float* kd = reinterpret_cast<const float*>(a.ws + p.off_k);
  double* dlam_acc = reinterpret_cast<double*>(a.ws + p.off_dlam);
  T* dx = static_cast<T*>(a.dx);
  T* dgl = static_cast<T*>(a.dgl);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cv = lane % kNvl, tcl = lane / kNvl;
  const int64_t BD = p.B * p.D;
  const int row0 = warp * kWarpSteps + tcl * kTc;
  const uint32_t box_tx = (uint32_t)p.tsteps * CH * sizeof(T);
  auto tile_at = [&](int64_t i) {  // this block's i-th tile (from the end in time)
    return decode_tile(i * gridDim.x + blockIdx.x, p.n_tiles_b, p.n_c_b, p.n_cg_b, CH, p.n_t, true);
  };
  auto issue = [&](int stage, const TileCoord& c) {
    unsigned char* dst = smem + (size_t)stage * NB * box_bytes<T>();
    const int t = (int)(c.tt * p.tsteps), d = (int)c.dbase, bb = (int)c.b;
    mbar_arrive_expect_tx(&bars[stage], NB * box_tx);
    tma_load_3d(dst, &a.tm_dh, &bars[stage], d, t, bb);
    tma_load_3d(dst + box_bytes<T>(), &a.tm_x, &bars[stage], d, t, bb);
    tma_load_3d(dst + 2 * box_bytes<T>(), &a.tm_gl, &bars[stage], d, t, bb);
    tma_load_3d(dst + 3 * box_bytes<T>(), &a.tm_gl, &bars[stage], (int)p.D + d, t, bb);
  };

  if (threadIdx.x == 0) {
    for (int j = 0; j < S; ++j) mbar_init(&bars[j], 1);
    fence_mbar_init();
  }
  if (threadIdx.x == 0) {
    const bool ok = __ldcg(&fh->tag) == p.tag && __ldcg(&fh->complete) == 1u;
    if (!ok) atomicOr(&fh->err, kErrWorkspace);
    s_flag = ok;
  }
  __syncthreads();
  if (!s_flag) return;  // no forward carries for this problem: write nothing
  if (threadIdx.x == 0) {
    for (int j = 0; j < S; ++j) {
      const TileCoord c = tile_at(j);
      if (c.tile < p.n_tiles_b) issue(j, c);
    }
  }
  float nk[VEC];
  {
    const TileCoord c = tile_at(0);
#pragma unroll
    for (int v = 0; v < VEC; ++v) nk[v] = 0.0f;
    if (c.tile < p.n_tiles_b && c.dbase + cv * VEC < p.D) load_f32<VEC>(kd + c.dbase + cv * VEC, nk);
  }

  for (int it = 0;; ++it) {
    const int stage = it % S;
    const int buf = it & 1;
    const TileCoord tc = tile_at(it);
    if (tc.tile >= p.n_tiles_b) break;
    const int64_t d0 = tc.dbase + cv * VEC;
    const bool ch_ok = d0 < p.D;
    const int64_t t0 = tc.tt * p.tsteps + row0;
    int64_t left = ch_ok ? p.L - t0 : 0;
    const int valid = (int)(left < 0 ? 0 : (left > kTc ? kTc : left));
    int lo = 0;
    if constexpr (VARLEN) {
      const int64_t head = row_start(a.lengths, tc.b, p.L) - t0;
      lo = (int)(head < 0 ? 0 : (head > kTc ? kTc : head));
    }
    float k[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) k[v] = nk[v];
    {
      const TileCoord c = tile_at(it + 1);
#pragma unroll
      for (int v = 0; v < VEC; ++v) nk[v] = 0.0f;
      if (c.tile < p.n_tiles_b && c.dbase + cv * VEC < p.D)
        load_f32<VEC>(kd + c.dbase + cv * VEC, nk);
    }

    // 1. the stage's rows, gates kept as E, r, i; chunk maps of both directions
    mbar_wait(&bars[stage], (uint32_t)(it / S) & 1u, &fh->err);
    const unsigned char* sb = smem + (size_t)stage * NB * box_bytes<T>();
    float gv[kTc][VEC], xv[kTc][VEC], ev[kTc][VEC], rv[kTc][VEC], iv[kTc][VEC];
    float A[VEC], U[VEC], W[VEC];
    {
      Raw rg[kTc], rx[kTc], rr[kTc], ri[kTc];
      lds_rows<IO>(sb, row0, cv, rg);
      lds_rows<IO>(sb + box_bytes<T>(), row0, cv, rx);
      lds_rows<IO>(sb + 2 * box_bytes<T>(), row0, cv, rr);
      lds_rows<IO>(sb + 3 * box_bytes<T>(), row0, cv, ri);
      if (valid == kTc && lo == 0)
        bwd_chunk<IO, M, true>(k, rg, rx, rr, ri, lo, valid, gv, xv, ev, rv, iv, A, U, W);
      else
        bwd_chunk<IO, M, false>(k, rg, rx, rr, ri, lo, valid, gv, xv, ev, rv, iv, A, U, W);
    }
    // 2. warp maps: h forwards (prefix), w backwards (suffix)
    float A2[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) A2[v] = A[v];
    float ea[VEC], eu[VEC], sa[VEC], sw[VEC];
    warp_prefix<VEC>(A, U, tcl, ea, eu);
    warp_suffix<VEC>(A2, W, tcl, sa, sw);
    if (tcl == kNtl - 1) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        s_wa[buf][warp][cv * VEC + v] = A[v];
        s_wu[buf][warp][cv * VEC + v] = U[v];
      }
    }
    if (tcl == 0) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) s_ww[buf][warp][cv * VEC + v] = W[v];
    }
    __syncthreads();  // the stage is read: refill it with the tile S ahead
    if (threadIdx.x == 0) {
      const TileCoord c = tile_at(it + S);
      if (c.tile < p.n_tiles_b) issue(stage, c);
    }

    // 3. warp 0, one lane per channel: warp prefix / suffix maps, the h carry
    //    from the forward, the w carry by look-back from the later tiles
    if (warp == 0) {
      const int ch = lane;
      const bool cval = tc.dbase + ch < p.D;
      float qa = 1.0f, qw = 0.0f;
      for (int w = p.nwarps - 1; w >= 0; --w) {  // suffix maps first: they read s_wa
        const float wA = s_wa[buf][w][ch], wW = s_ww[buf][w][ch];
        s_ws[buf][w][ch] = qa;
        s_ww[buf][w][ch] = qw;
        qw = fmaf(wA, qw, wW);
        qa *= wA;
      }
      float pa = 1.0f, pu = 0.0f;
      for (int w = 0; w < p.nwarps; ++w) {
        const float wA = s_wa[buf][w][ch], wU = s_wu[buf][w][ch];
        s_wa[buf][w][ch] = pa;
        s_wu[buf][w][ch] = pu;
        pu = fmaf(wA, pu, wU);
        pa *= wA;
      }
      float hc = 0.0f, wc = 0.0f;
      if (cval) {
        const int64_t rec = tc.tt * BD + tc.b * p.D + tc.dbase + ch;
        if (tc.tt > 0)
          hc = __ldcg(&fpre[rec - BD]);
        else if (a.h0 != nullptr)
          hc = a.h0[tc.b * p.D + tc.dbase + ch];
        if (tc.tt == p.n_t - 1) {
          if (a.dh_last != nullptr) wc = a.dh_last[tc.b * p.D + tc.dbase + ch];
        } else {
          st_record(&agg[rec], pack_agg(qa, qw));
          wc = lookback(agg + rec + BD, pre + rec + BD, BD, p.n_t - 1 - tc.tt, &fh->err);
        }
        const float incl = fmaf(qa, wc, qw);  // w at the tile's first step
        st_record(&pre[rec], __float_as_uint(incl));
        if (tc.tt == 0 && a.dh0 != nullptr) a.dh0[tc.b * p.D + tc.dbase + ch] = incl;
      }
      s_hc[buf][ch] = hc;
      s_wc[buf][ch] = wc;
    }
    __syncthreads();

    // 4. g backwards through the chunk, then the gradients forwards with h_{t-1}
    float hs[VEC], wn[VEC], dlr[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const int c = cv * VEC + v;
      hs[v] = fmaf(ea[v], fmaf(s_wa[buf][warp][c], s_hc[buf][c], s_wu[buf][warp][c]), eu[v]);
      wn[v] = fmaf(sa[v], fmaf(s_ws[buf][warp][c], s_wc[buf][c], s_ww[buf][warp][c]), sw[v]);
      dlr[v] = 0.0f;
    }
#pragma unroll
    for (int s = kTc - 1; s >= 0; --s) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        const float g = gv[s][v] + wn[v];
        gv[s][v] = g;
        wn[v] = (1.0f + ev[s][v]) * g;
      }
    }
    const int64_t row = tc.b * p.L + t0;
    T* pdx = dx + row * p.D + d0;
    T* pdg = dgl + row * 2 * p.D + d0;
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      float ox[VEC], orho[VEC], oiota[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        const float e = ev[s][v], r = rv[s][v], i = iv[s][v], g = gv[s][v];
        const float alpha = 1.0f + e;
        const float q = -e * (2.0f + e);
        float beta, uu, c2;  // beta = n i, u = beta x, c2 = alpha u / q = alpha i x / n
        M::norm_terms(q, i, xv[s][v], alpha, beta, uu, c2);
        const float dl = g * alpha * (hs[v] - c2);
        orho[v] = dl * k[v] * (r - r * r);
        oiota[v] = g * uu * (1.0f - i);
        ox[v] = g * beta;
        dlr[v] = fmaf(dl, r, dlr[v]);
        hs[v] = fmaf(alpha, hs[v], uu);
      }
      if (s >= lo && s < valid) {
        IO::store(pdx + s * p.D, ox);
        IO::store(pdg + s * 2 * p.D, orho);
        IO::store(pdg + s * 2 * p.D + p.D, oiota);
      }
    }
    // 5. dLambda: sum over the warp's time lanes, one float64 add per channel
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
#pragma unroll
      for (int off = 1; off < kNtl; off <<= 1) dlr[v] += __shfl_down_sync(kFull, dlr[v], off * kNvl);
    }
    if (tcl == 0 && ch_ok) {
      double* acc = dlam_acc + (tc.b % kStripes) * p.D + d0;
#pragma unroll
      for (int v = 0; v < VEC; ++v) atomicAdd(acc + v, (double)dlr[v]);
    }
  }
  // The last block out turns the partial sums into dLambda.
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_flag = (atomicAdd(&bh->exited, 1u) == gridDim.x - 1) ? 2 : 1;
  }
  __syncthreads();
  if (s_flag == 2) {
    __threadfence();
    for (int64_t d = threadIdx.x; d < p.D; d += blockDim.x) {
      double sum = 0.0;
      for (int st = 0; st < kStripes; ++st) sum += __ldcg(&dlam_acc[st * p.D + d]);
      const double lam = (double)a.lambda[d];
      const double sig = 1.0 / (1.0 + exp(-lam));  // d softplus / d Lambda
      a.dlambda[d] = (float)(-(double)p.c * sig * sum);
    }
  }
}

// ------------------------------------------------------------ recurrent step
//
// h_t = alpha h_prev + beta x for B rows of D channels. A persistent grid: a
// block covers blockDim.x channel vectors and computes k = -c softplus(Lambda)
// for them once; each thread then walks rows ROWS at a time, with a stride of
// the grid's row threads, loading the next rows' inputs before the current
// rows' arithmetic so that every thread keeps loads in flight.

constexpr int kStepBlocksPerSm = 3;

template <typename T, int VEC, class M, int ROWS>
__global__ void __launch_bounds__(256, kStepBlocksPerSm) step_kernel(const StepArgs a) {
  using IO = Io<T, VEC>;
  __shared__ float s_k[64 * 8];
  const int64_t vg = blockIdx.x % a.n_vgroups;
  const int64_t rg = blockIdx.x / a.n_vgroups;
  const int64_t n_rg = gridDim.x / a.n_vgroups;  // the grid launches whole channel groups
  const int64_t dblock = vg * blockDim.x * VEC;
  const int tid = threadIdx.y * blockDim.x + threadIdx.x;
  for (int j = tid; j < (int)blockDim.x * VEC; j += blockDim.x * blockDim.y)
    if (dblock + j < a.D) s_k[j] = decay_rate(a.c, a.lambda[dblock + j]);
  __syncthreads();
  const int64_t d0 = dblock + threadIdx.x * VEC;
  if (d0 >= a.D) return;
  float k[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) k[v] = s_k[threadIdx.x * VEC + v];
  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);
  const int64_t rstride = n_rg * blockDim.y * ROWS;  // rows the grid takes per step of the walk
  float hp[ROWS][VEC], xv[ROWS][VEC], rv[ROWS][VEC], iv[ROWS][VEC];
  auto load = [&](int64_t r0) {
#pragma unroll
    for (int r = 0; r < ROWS; ++r) {
      const int64_t bb = r0 + r;
      if (bb < a.B) {
        load_f32<VEC>(a.h_prev + bb * a.D + d0, hp[r]);
        IO::unpack(IO::load_raw(x + bb * a.D + d0), xv[r]);
        IO::unpack(IO::load_raw(gl + bb * 2 * a.D + d0), rv[r]);
        IO::unpack(IO::load_raw(gl + bb * 2 * a.D + a.D + d0), iv[r]);
      }
    }
  };
  int64_t r0 = (rg * blockDim.y + threadIdx.y) * ROWS;
  if (r0 < a.B) load(r0);
  for (; r0 < a.B; r0 += rstride) {
    float ch[ROWS][VEC], cx[ROWS][VEC], cr[ROWS][VEC], ci[ROWS][VEC];
#pragma unroll
    for (int r = 0; r < ROWS; ++r) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        ch[r][v] = hp[r][v];
        cx[r][v] = xv[r][v];
        cr[r][v] = rv[r][v];
        ci[r][v] = iv[r][v];
      }
    }
    if (r0 + rstride < a.B) load(r0 + rstride);  // in flight during this rows' arithmetic
#pragma unroll
    for (int r = 0; r < ROWS; ++r) {
      const int64_t bb = r0 + r;
      if (bb < a.B) {
        float out[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          const float rr = M::sigmoid(cr[r][v]);
          const float i = M::sigmoid(ci[r][v]);
          const float e = M::expm1_any(k[v] * rr);
          out[v] = fmaf(1.0f + e, ch[r][v], M::sqrt(-e * (2.0f + e)) * i * cx[r][v]);
        }
#pragma unroll
        for (int j = 0; j < VEC; j += 4)
          __stcs(reinterpret_cast<float4*>(a.h_t + bb * a.D + d0 + j),
                 make_float4(out[j], out[j + 1], out[j + 2], out[j + 3]));
      }
    }
  }
}

// ------------------------------------------------------- K recurrent steps
//
// h_j = alpha_j h_{j-1} + beta_j x_j for j = 1..K and every (row, channel), from
// h_0 = h_prev: a thread owns VEC channels of one row and walks its K steps
// serially with the state in float32 registers, whatever the state dtype in
// memory (a bfloat16 state is rounded once, when it is stored). The loads of
// kStepsAhead steps are issued before the first of them is used.

struct StepsArgs {
  int64_t B, K, D;
  float c;
  const void* h_prev;  // (B, D), state dtype
  const void* x;       // (B, K, D), io dtype
  const void* gl;      // (B, K, 2D), io dtype
  const float* lambda;
  void* h_out;         // (B, D), state dtype
  void* h_seq;         // (B, K, D), io dtype, or NULL
};

constexpr int kStepsAhead = 4;

template <typename S, int VEC>
__device__ __forceinline__ void load_state(const S* p, float (&h)[VEC]) {
  if constexpr (sizeof(S) == 4)
    load_f32<VEC>(reinterpret_cast<const float*>(p), h);
  else
    Io<__nv_bfloat16, VEC>::unpack(Io<__nv_bfloat16, VEC>::load_raw(p), h);
}
template <typename S, int VEC>
__device__ __forceinline__ void store_state(S* p, const float (&h)[VEC]) {
  if constexpr (sizeof(S) == 4) {
#pragma unroll
    for (int j = 0; j < VEC; j += 4)
      *reinterpret_cast<float4*>(reinterpret_cast<float*>(p) + j) =
          make_float4(h[j], h[j + 1], h[j + 2], h[j + 3]);
  } else {
    Io<__nv_bfloat16, VEC>::store(p, h);
  }
}

template <typename T, typename S, int VEC, class M>
__global__ void __launch_bounds__(256) steps_kernel(const StepsArgs a) {
  using IO = Io<T, VEC>;
  using Raw = typename IO::Raw;
  const int64_t nv = a.D / VEC;
  const int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (idx >= a.B * nv) return;
  const int64_t b = idx / nv;
  const int64_t d0 = (idx - b * nv) * VEC;
  float k[VEC], h[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) k[v] = decay_rate(a.c, a.lambda[d0 + v]);
  load_state<S, VEC>(static_cast<const S*>(a.h_prev) + b * a.D + d0, h);
  const T* x = static_cast<const T*>(a.x) + b * a.K * a.D + d0;
  const T* gl = static_cast<const T*>(a.gl) + b * a.K * 2 * a.D + d0;
  T* hs = a.h_seq != nullptr ? static_cast<T*>(a.h_seq) + b * a.K * a.D + d0 : nullptr;
  for (int64_t j0 = 0; j0 < a.K; j0 += kStepsAhead) {
    Raw rx[kStepsAhead], rr[kStepsAhead], ri[kStepsAhead];
#pragma unroll
    for (int u = 0; u < kStepsAhead; ++u) {
      const int64_t j = j0 + u;
      if (j < a.K) {
        rx[u] = IO::load_raw(x + j * a.D);
        rr[u] = IO::load_raw(gl + j * 2 * a.D);
        ri[u] = IO::load_raw(gl + j * 2 * a.D + a.D);
      }
    }
#pragma unroll
    for (int u = 0; u < kStepsAhead; ++u) {
      const int64_t j = j0 + u;
      if (j < a.K) {
        float xv[VEC], rv[VEC], iv[VEC];
        IO::unpack(rx[u], xv);
        IO::unpack(rr[u], rv);
        IO::unpack(ri[u], iv);
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          const float r = M::sigmoid(rv[v]);
          const float i = M::sigmoid(iv[v]);
          const float e = M::expm1_any(k[v] * r);
          h[v] = fmaf(1.0f + e, h[v], M::sqrt(-e * (2.0f + e)) * i * xv[v]);
        }
        if (hs != nullptr) IO::store(hs + j * a.D, h);
      }
    }
  }
  store_state<S, VEC>(static_cast<S*>(a.h_out) + b * a.D + d0, h);
}

// ------------------------------------------------------------ bounded-wait test

__global__ void selftest_wait_kernel(const uint32_t* flag, uint32_t* err, uint64_t timeout_ns) {
  (void)wait_word(flag, err, timeout_ns);
}

}  // namespace blr
