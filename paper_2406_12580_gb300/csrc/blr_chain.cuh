// Chained single-pass forward scan: the BD-LRU forward for problems with few
// (batch row, channel group) chains and long sequences, reading every input
// once and writing every output once.
//
// The path is bfloat16 I/O. A tile is kChainTile consecutive steps of one
// chain (64 bfloat16 channels of one batch row, a 128-byte row segment; a
// lane owns 2 channels as one float pair). Tiles are numbered
// time-major (tile = time block * chains + chain); block j of a cooperative
// grid of G resident blocks (one per SM) takes tiles j, j + G, j + 2G, ..., so
// a tile only ever waits on tiles of smaller number. The block's warps have
// fixed roles and hand tiles on through mbarriers:
//   producer (1 warp): loads tile n's x, rho and iota boxes into stage n % S of
//      a shared-memory ring by TMA once the stage is free, and writes the
//      tile's per-channel decay constants k = -c softplus(Lambda) beside it;
//   compute (kChainWarps warps, a slice of kChainSlice steps each): pass A of
//      tile n evaluates the gates of Sec. 3.2 for the slice from the stage
//      (which is then released), folds it serially from a zero state (hl_t,
//      and am_t = the product of the alphas so far minus one, so that h_t =
//      hl_t + (1 + am_t) h_start), publishes the slice's map (A - 1, U) and
//      parks the per-step hl_t, am_t in the block's tensor memory (TMEM: the
//      warp's 32 lanes x 2 kChainSlice VEC columns of a slot, written 16
//      columns at a time as the fold advances), off the register file until
//      pass C needs them.
//      Then pass C of tile n - kChainLag, whose entering states the scanners
//      have found meanwhile: h_t = hl_t + (1 + am_t) h_start is written to global
//      memory from registers (coalesced 128-byte rows), with the kept states
//      the backward starts from;
//   scanners (kChainScanners warps, tiles in turn): compose the slice maps into the
//      tile's map (the operator of Sec. 3.3, (a2, u2) . (a1, u1) = (a2 a1,
//      a2 u1 + u2)), publish it, find the state entering the tile with
//      a decoupled look-back over the records of the tiles before it in the
//      same chain, publish the state after the tile, and hand every slice its
//      starting state.
// The look-back's round trips to L2 thus overlap kChainLag tiles' arithmetic
// instead of stalling it, and the ring keeps several tiles' loads in flight.
//
// Products of alphas are carried as their difference from one (m = A - 1):
// with slow decays a product of a few alphas lies within 1e-3 of one, where a
// float32 holds only a few significant digits of 1 - A, which the large states
// of slow decays then multiply. A map h -> A h + U is applied as
// (m h + h) + U, and two maps compose as m = m1 + m2 + m1 m2.
//
// Records validate themselves: a record is one relaxed 32- or 64-bit store of
// a value that is never the all-ones pattern the records are filled with
// before the call (A - 1 lies in (-1, 0]; a float state is never that NaN).
#pragma once

#include "blr_seq.cuh"

namespace blr {

constexpr int kChainStages = 4;             // ring stages per block
constexpr int kChainLag = 3;                // pass C runs this many tiles behind pass A
constexpr int kChainSlots = kChainLag + 1;  // slice-map, starting-state and TMEM slots
constexpr uint32_t kChainTmemCols = 512;    // TMEM columns the block allocates (all of them)
constexpr int kChainScanners = 3;
// Predecessors read per look-back round trip. By the time a tile looks back,
// its nearest predecessor has usually published its inclusive value, so a
// short window saves loads (measured on 8 x 32768 x 512: windows of 1-2 gave
// the fastest forward and backward, 6 was 3 % slower).
constexpr int kChainWindow = 2;
constexpr int kChainThreads = (kChainWarps + kChainScanners + 1) * 32;
// Registers per thread: each of the SM's 4 schedulers holds a quarter of the
// 65536 registers and a quarter of the warps (rounded up); rounded down to the
// allocation granule of 8.
constexpr int kChainMaxRegs = (16384 / (((kChainThreads / 32 + 3) / 4) * 32)) / 8 * 8;

struct ChainFwdArgs {
  CUtensorMap tm_x;
  CUtensorMap tm_r;
  CUtensorMap tm_i;
  Plan p;
  const float* lambda;
  const float* h0;
  void* h;  // (B, L, D) io dtype, or NULL (kept states and h_last only)
  float* h_last;
  unsigned char* ws;
};

template <typename T, int VEC>
__host__ __device__ constexpr uint32_t chain_box_bytes() {
  return (uint32_t)(kChainTile * 32 * VEC * sizeof(T));
}

// Shared memory, in this order from a 128-byte aligned base: the ring
// (stages of 3 boxes), the stages' decay constants (k, k/2) and POLY flags, the
// slots' slice maps (which the scanner overwrites with the slices' starting
// states, in .x) and tile coordinates, the tensor-memory base address, and the
// mbarriers (full and empty per stage, maps-ready and carry-ready per slot).
// Every region starts on a 16-byte boundary.
template <typename T, int VEC>
struct ChainSmem {
  static constexpr int CHW = 32 * VEC;
  static constexpr size_t up(size_t v) { return (v + 15) / 16 * 16; }
  static constexpr size_t ring = (size_t)kChainStages * 3 * chain_box_bytes<T, VEC>();
  static constexpr size_t rates = up(ring);  // float2 [S][CHW]
  static constexpr size_t poly = up(rates + (size_t)kChainStages * CHW * sizeof(float2));  // int [S]
  static constexpr size_t maps = up(poly + (size_t)kChainStages * sizeof(int));  // float2 [M][W][CHW]
  static constexpr size_t meta = up(maps + (size_t)kChainSlots * kChainWarps * CHW * sizeof(float2));  // int4 [M]
  static constexpr size_t tmem = up(meta + (size_t)kChainSlots * sizeof(int4));  // uint32: TMEM base
  static constexpr size_t bars = up(tmem + sizeof(uint32_t));
  static constexpr size_t end = bars + (size_t)(2 * kChainStages + 2 * kChainSlots) * sizeof(uint64_t);
  static constexpr size_t bytes = end + 128;  // slack for the alignment of the base
  static_assert(rates % 16 == 0 && poly % 16 == 0 && maps % 16 == 0 && meta % 16 == 0 &&
                tmem % 16 == 0 && bars % 16 == 0, "");
};

// The map h -> (1 + m) h + U applied to h, and the composition of the minus-one
// parts of two maps' products.
__device__ __forceinline__ float map_apply(float m, float h, float U) { return fmaf(m, h, h) + U; }
__device__ __forceinline__ float2 map_apply2(float2 m, float2 h, float2 U) {
  return __fadd2_rn(__ffma2_rn(m, h, h), U);
}
__device__ __forceinline__ float m_compose(float m1, float m2) { return fmaf(m1, m2, m1 + m2); }

// Pass A for a bfloat16 lane (two channels, carried as one float2 so that the
// multiply-adds run as packed pairs), the 4 rows of its warp's slice whose
// states fill 16 TMEM columns: the gates of the rows (as the serial forward
// evaluates them, GatesFast), then the fold continued from (H, M), the state
// and the product of alphas minus one after the slice's earlier rows (zero at
// its start). Row r's states go to park[4r, 4r + 4) as (H.x, M.x, H.y, M.y).
template <bool POLY>
__device__ __forceinline__ void chain_fold_part_bf16x2(const unsigned char* lb, float2 kh, float2& H,
                                                       float2& M, float (&park)[16]) {
  constexpr int QS = 4;
  constexpr uint32_t ROWB = 128;
  constexpr uint32_t BOX = kChainTile * ROWB;
  float2 hl[QS], am[QS];
#pragma unroll
  for (int s = 0; s < QS; ++s) {
    const float2 hx = bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + s * ROWB), kBf2Half);
    const float2 hr = bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + BOX + s * ROWB), kBf2Half);
    const float2 hi = bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + 2 * BOX + s * ROWB), kBf2Half);
    // l = kh tanh(rho/2) + kh, e = e^l - 1
    const float2 e = expm1_neg2<POLY>(__ffma2_rn(kh, tanh2(hr), kh));
    am[s] = e;
    // 1 - alpha^2 = -e (e + 2); u = sqrt(1 - alpha^2) i x with i x = (x/2) tanh(iota/2) + x/2
    const float2 m2 = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));
    hl[s] = __fmul2_rn(make_float2(sqrt_approx(-m2.x), sqrt_approx(-m2.y)),
                       __ffma2_rn(hx, tanh2(hi), hx));
  }
#pragma unroll
  for (int s = 0; s < QS; ++s) {
    const float2 alpha = __fadd2_rn(f2(1.0f), am[s]);
    H = __ffma2_rn(alpha, H, hl[s]);
    M = __ffma2_rn(alpha, M, am[s]);  // alpha (1 + M) - 1
    park[4 * s] = H.x;
    park[4 * s + 1] = M.x;
    park[4 * s + 2] = H.y;
    park[4 * s + 3] = M.y;
  }
}

// ---------------------------------------------------------------- look-back
//
// One channel's walk over the tile's nprev predecessors, nearest first: the
// q-th has its records at inc[q * step] and agg[q * step] (step = -BD when
// the predecessors are the earlier time blocks, as in the forward; +BD when
// they are the later ones, as in the backward). kChainWindow predecessors are
// read in one round trip; the walk folds aggregates until it meets a published
// state. The farthest predecessor publishes only its state, so every walk ends.

struct ChainWindow {
  uint32_t in[kChainWindow];
  unsigned long long ag[kChainWindow];
};

__device__ __forceinline__ void chain_window_load(const unsigned long long* agg, const uint32_t* inc,
                                                  int64_t step, int64_t q0, int64_t nprev,
                                                  ChainWindow& w) {
#pragma unroll
  for (int q = 0; q < kChainWindow; ++q) {
    w.in[q] = kEmpty;
    w.ag[q] = ~0ull;
    if (q0 + q < nprev) {
      w.in[q] = ld_record(inc + (q0 + q) * step);
      w.ag[q] = ld_record(agg + (q0 + q) * step);
    }
  }
}

// The value entering the tile (its predecessors' state, or adjoint, carried
// through them), starting from the window `w` already loaded for q0 = 0. On an
// expired wait (recorded in *err) it returns what it has.
__device__ __forceinline__ float chain_walk(const unsigned long long* agg, const uint32_t* inc,
                                           int64_t step, int64_t nprev, uint32_t* err, ChainWindow& w) {
  float em = 0.0f, eu = 0.0f;  // the fold of the aggregates walked so far: h -> (1 + em) h + eu
  int64_t q0 = 0;
  for (;;) {
    int adv = kChainWindow;
    bool open = true, wait = false;
#pragma unroll
    for (int q = 0; q < kChainWindow; ++q) {
      if (open) {
        if (w.in[q] != kEmpty) return map_apply(em, __uint_as_float(w.in[q]), eu);
        if (agg_empty(w.ag[q])) {  // nothing published yet: wait for it, then re-read from it
          open = false;
          wait = true;
          adv = q;
        } else {
          eu = map_apply(em, __uint_as_float((uint32_t)(w.ag[q] >> 32)), eu);
          em = m_compose(em, __uint_as_float((uint32_t)w.ag[q]));
        }
      }
    }
    if (q0 + adv >= nprev) return eu;  // no predecessor left (cannot happen: the farthest publishes its state)
    if (wait && !wait_record(inc + (q0 + adv) * step, agg + (q0 + adv) * step, err, kWaitTimeoutNs))
      return eu;  // the wait expired (recorded): finish with what is known
    q0 += adv;
    chain_window_load(agg, inc, step, q0, nprev, w);
  }
}

// ------------------------------------------------------------------- kernel

template <typename T, class M, int VEC, int RB>
__global__ void __maxnreg__(kChainMaxRegs) chain_fwd_kernel(const __grid_constant__ ChainFwdArgs a) {
  using IO = Io<T, VEC>;
  using G = typename GatePolicy<M>::type;
  using SM = ChainSmem<T, VEC>;
  constexpr int CHW = 32 * VEC;
  constexpr int NB = 3;  // boxes per stage: x, rho, iota
  constexpr int S = kChainStages, NW = kChainWarps, TS = kChainSlice, MS = kChainSlots;
  constexpr int LAG = kChainLag;
  constexpr uint32_t ROWB = CHW * sizeof(T);
  constexpr uint32_t BOX = chain_box_bytes<T, VEC>();
  static_assert(VEC == 2 && G::kHalfInputs, "the chained kernels are the bfloat16 path");
  // A lane's states of one slice fill NP parts of 16 TMEM columns (QS rows each).
  constexpr int QS = 16 / (2 * VEC), NP = TS / QS;
  static_assert(QS * 2 * VEC == 16 && NP * QS == TS && NP <= 4, "slices of whole 16-column parts");
  static_assert(RB % TS == 0 || TS % RB == 0, "kept states fall on slice rows");
  static_assert(NW % 4 == 0 && (NW / 4) * 16 * NP * MS <= kChainTmemCols, "TMEM slots");
  const Plan& p = a.p;
  extern __shared__ unsigned char chain_smem[];
  unsigned char* base = align128(chain_smem);
  float2* rates = reinterpret_cast<float2*>(base + SM::rates);  // [S][CHW]: (k, k/2)
  int* polys = reinterpret_cast<int*>(base + SM::poly);         // [S]
  float2* maps = reinterpret_cast<float2*>(base + SM::maps);    // [MS][NW][CHW]
  int4* meta = reinterpret_cast<int4*>(base + SM::meta);        // [MS]: (time block, row, group)
  uint32_t* tslot = reinterpret_cast<uint32_t*>(base + SM::tmem);
  uint64_t* full = reinterpret_cast<uint64_t*>(base + SM::bars);
  uint64_t* empty = full + S;
  uint64_t* maps_ready = empty + S;
  uint64_t* carry_ready = maps_ready + MS;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t C = p.n_chain;
  const int64_t n_g = (p.D + CHW - 1) / CHW;
  const int64_t BD = p.B * p.D;
  const int64_t n_tiles = p.n_tc * C;
  const int64_t G_ = gridDim.x;
  const int64_t n_my = blockIdx.x < n_tiles ? (n_tiles - blockIdx.x + G_ - 1) / G_ : 0;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  uint32_t* err = &fh->err;

  // The backward of these problems is the segmented one: tag the workspace
  // for it and restart its bookkeeping.
  if (blockIdx.x == 0 && warp == 0) seq_reset_workspace(a.ws, p, seg_tag(p.tag), lane);
  if (warp == 0) {  // the block's TMEM, freed by this warp after the final barrier
    __syncwarp();
    tmem_alloc(tslot, kChainTmemCols);
    tmem_fence_before_sync();
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], NW * 32);
    }
    for (int m = 0; m < MS; ++m) {
      mbar_init(&maps_ready[m], NW * 32);
      mbar_init(&carry_ready[m], 32);
    }
    fence_mbar_init();
  }
  __syncthreads();  // the roles part here and meet again at the end

  // Tile n of this block: (time block, batch row, channel group). Tile and
  // chain counts stay below 2^31 (checked on the host): 32-bit division.
  const uint32_t C32 = (uint32_t)C, ng32 = (uint32_t)n_g;
  auto coord = [&](int64_t n) {
    const uint32_t tile = (uint32_t)(blockIdx.x + n * G_);
    const uint32_t tb = tile / C32, chain = tile - tb * C32;
    const uint32_t b = chain / ng32;
    return make_int4((int)tb, (int)b, (int)(chain - b * ng32), 0);
  };

  if (warp == NW + kChainScanners) {
    // ---------------------------------------------------------- producer
    // The decay constants of tile n + 1 are evaluated (their Lambda loads in
    // flight) while the stage for tile n is awaited.
    float k[VEC], kh[VEC], nk[VEC], nkh[VEC];
    int poly = 0, npoly = 0;
    if (n_my > 0) {
      const int4 c = coord(0);
      const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
      npoly = seq_rates<VEC>(a.lambda, p.c, d0, d0 < p.D, nk, nkh) ? 1 : 0;
    }
    for (int64_t n = 0; n < n_my; ++n) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        k[v] = nk[v];
        kh[v] = nkh[v];
      }
      poly = npoly;
      if (n + 1 < n_my) {
        const int4 c = coord(n + 1);
        const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
        npoly = seq_rates<VEC>(a.lambda, p.c, d0, d0 < p.D, nk, nkh) ? 1 : 0;
      }
      const int s = (int)(n % S);
      if (n >= S) mbar_wait(&empty[s], (uint32_t)(n / S - 1) & 1u, err);  // tile n - S released it
#pragma unroll
      for (int v = 0; v < VEC; ++v) rates[s * CHW + lane * VEC + v] = make_float2(k[v], kh[v]);
      if (lane == 0) polys[s] = poly;
      __syncwarp();
      if (lane == 0) {  // the arrival releases the rates above with the stage
        const int4 c = coord(n);
        unsigned char* dst = base + (size_t)s * NB * BOX;
        const int t = c.x * kChainTile, cd = c.z * CHW, cb = c.y;
        mbar_arrive_expect_tx(&full[s], NB * BOX);
        tma_load_3d(dst, &a.tm_x, &full[s], cd, t, cb);
        tma_load_3d(dst + BOX, &a.tm_r, &full[s], cd, t, cb);
        tma_load_3d(dst + 2 * BOX, &a.tm_i, &full[s], cd, t, cb);
      }
    }
  } else if (warp >= NW) {
    // ---------------------------------------------------------- scanners
    unsigned long long* agg = reinterpret_cast<unsigned long long*>(a.ws + p.off_cagg);
    uint32_t* inc = reinterpret_cast<uint32_t*>(a.ws + p.off_cinc);
    for (int64_t n = warp - NW; n < n_my; n += kChainScanners) {
      const int m = (int)(n % MS);
      const int4 c = coord(n);
      const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
      const bool ch_ok = d0 < p.D;
      mbar_wait(&maps_ready[m], (uint32_t)(n / MS) & 1u, err);
      float TM[VEC], TU[VEC], hs[VEC];  // the tile's map h -> (1 + TM) h + TU
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        TM[v] = 0.0f;
        TU[v] = 0.0f;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
          const float2 e = maps[(m * NW + w) * CHW + lane * VEC + v];
          TU[v] = map_apply(e.x, TU[v], e.y);
          TM[v] = m_compose(TM[v], e.x);
        }
        hs[v] = 0.0f;
      }
      if (ch_ok) {
        const int64_t ch0 = (int64_t)c.y * p.D + d0;  // the channel's records of time block 0
        const int64_t rec = (int64_t)c.x * BD + ch0;
        if (c.x == 0) {
          if (a.h0 != nullptr) {
#pragma unroll
            for (int v = 0; v < VEC; ++v) hs[v] = a.h0[ch0 + v];
          }
        } else {
#pragma unroll
          for (int v = 0; v < VEC; ++v) st_record(&agg[rec + v], pack_agg(TM[v], TU[v]));
          // predecessors: time blocks c.x - 1, c.x - 2, ..., 0
          const int64_t near = rec - BD;
          ChainWindow win[VEC];
#pragma unroll
          for (int v = 0; v < VEC; ++v) chain_window_load(agg + near + v, inc + near + v, -BD, 0, c.x, win[v]);
#pragma unroll
          for (int v = 0; v < VEC; ++v) hs[v] = chain_walk(agg + near + v, inc + near + v, -BD, c.x, err, win[v]);
        }
#pragma unroll
        for (int v = 0; v < VEC; ++v) st_record(&inc[rec + v], __float_as_uint(map_apply(TM[v], hs[v], TU[v])));
      }
      // every slice's starting state: the carry through the slices before it,
      // written over the slice's map
#pragma unroll
      for (int w = 0; w < NW; ++w) {
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          float2* e = &maps[(m * NW + w) * CHW + lane * VEC + v];
          const float2 mw = *e;
          e->x = hs[v];
          hs[v] = map_apply(mw.x, hs[v], mw.y);
        }
      }
      if (lane == 0) meta[m] = c;
      mbar_arrive(&carry_ready[m]);
    }
  } else {
    // ---------------------------------------------------------- compute
    // Pass A of tile n parks the slice's per-step states (hl_t, ap_t) in TMEM
    // slot n % MS of this warp's lanes and columns; pass C of tile n - LAG
    // takes them back once its starting state has arrived. Each iteration runs
    // C first, so that A's park store has a whole iteration to complete before
    // the next A waits for it.
    tmem_fence_after_sync();
    constexpr uint32_t kWarpCols = 16 * NP;
    constexpr uint32_t kSlotCols = (NW / 4) * kWarpCols;
    const uint32_t tq = *tslot + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(warp >> 2) * kWarpCols;
    T* h = static_cast<T*>(a.h);
    float* kept = reinterpret_cast<float*>(a.ws + p.off_skept);
    const uint32_t loff = warp * TS * ROWB + lane * VEC * sizeof(T);  // this lane's first row
    const uint32_t nmy = (uint32_t)n_my;  // below 2^31 (the tile count is)
    for (uint32_t n = 0; n < nmy + LAG; ++n) {
      if (n >= LAG) {
        // ---- C: tile n - LAG's states from the starting state its scanner handed over
        // its parked states first (ready since its pass A), then its starting state
        const uint32_t q = n - LAG;
        const uint32_t m = q % MS;
        uint32_t pr[NP][16];
        __syncwarp();  // tcgen05 accesses are warp-collective
#pragma unroll
        for (int part = 0; part < NP; ++part) tmem_ld16_start(tq + m * kSlotCols + part * 16, pr[part]);
        mbar_wait(&carry_ready[m], (q / MS) & 1u, err);
        const int4 c = meta[m];
        float hs[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) hs[v] = maps[(m * NW + warp) * CHW + lane * VEC + v].x;
        __syncwarp();
#pragma unroll
        for (int part = 0; part < NP; ++part) tmem_ld_wait(pr[part]);
        float out[TS][VEC];
#pragma unroll
        for (int r = 0; r < TS; ++r) {
          const uint32_t* pk = pr[r / QS];
          const int r0 = r % QS;
          const float2 o = map_apply2(
              make_float2(__uint_as_float(pk[4 * r0 + 1]), __uint_as_float(pk[4 * r0 + 3])),
              make_float2(hs[0], hs[1]),
              make_float2(__uint_as_float(pk[4 * r0]), __uint_as_float(pk[4 * r0 + 2])));
          out[r][0] = o.x;
          out[r][1] = o.y;
        }
        const uint32_t d0 = (uint32_t)c.z * CHW + lane * VEC;  // D < 2^24
        const uint32_t t0 = (uint32_t)c.x * kChainTile + warp * TS;  // L < 2^31
        if (d0 < p.D && t0 < p.L) {
          const int rows = p.L - t0 < TS ? (int)(p.L - t0) : TS;
          const int64_t row0 = (int64_t)c.y * p.D + d0;  // (batch row, channel) offset of a state
          if (h != nullptr) {
            T* ph = h + ((int64_t)c.y * p.L + t0) * p.D + d0;
            if (rows == TS) {
#pragma unroll
              for (int r = 0; r < TS; ++r) {
                IO::store(ph, out[r]);
                ph += p.D;
              }
            } else {
#pragma unroll
              for (int r = 0; r < TS; ++r) {
                if (r < rows) IO::store(ph, out[r]);
                ph += p.D;
              }
            }
          }
          // kept states: the rows that end a block of RB steps (a slice's last
          // row, or every RB-th row of a slice that spans several blocks)
          if constexpr (TS % RB == 0) {
#pragma unroll
            for (int r = RB - 1; r < TS; r += RB) {
              const int64_t mk = (t0 + r + 1) / RB - 1;
              if (r < rows && mk < p.n_carry) {
#pragma unroll
                for (int v = 0; v < VEC; ++v) kept[mk * BD + row0 + v] = out[r][v];
              }
            }
          } else if (rows == TS && (t0 + TS) % RB == 0) {
            const int64_t mk = (t0 + TS) / RB - 1;
            if (mk < p.n_carry) {
#pragma unroll
              for (int v = 0; v < VEC; ++v) kept[mk * BD + row0 + v] = out[TS - 1][v];
            }
          }
          if (a.h_last != nullptr && t0 + rows == p.L) {
            float last[VEC];  // out[rows - 1], selected without indexing by a variable
#pragma unroll
            for (int v = 0; v < VEC; ++v) last[v] = out[0][v];
#pragma unroll
            for (int r = 1; r < TS; ++r) {
#pragma unroll
              for (int v = 0; v < VEC; ++v) last[v] = r < rows ? out[r][v] : last[v];
            }
#pragma unroll
            for (int v = 0; v < VEC; ++v) a.h_last[row0 + v] = last[v];
          }
        }
      }
      if (n < nmy) {
        // ---- A: tile n's gates and slice fold, parked 16 columns at a time;
        // the stage is free again afterwards
        const uint32_t s = n % S, m = n % MS;
        tmem_wait_st();  // the previous tile's park stores, before a later load of their slot
        mbar_wait(&full[s], (n / S) & 1u, err);
        const unsigned char* lb = base + s * (NB * BOX) + loff;
        const bool poly = polys[s] != 0;
        const float2 r0 = rates[s * CHW + lane * 2], r1 = rates[s * CHW + lane * 2 + 1];
        const float2 kh = make_float2(r0.y, r1.y);
        float2 H = make_float2(0.0f, 0.0f), Am = make_float2(0.0f, 0.0f);
#pragma unroll
        for (int part = 0; part < NP; ++part) {
          float park[16];
          if (poly)
            chain_fold_part_bf16x2<true>(lb + part * QS * ROWB, kh, H, Am, park);
          else
            chain_fold_part_bf16x2<false>(lb + part * QS * ROWB, kh, H, Am, park);
          __syncwarp();
          tmem_st16(tq + m * kSlotCols + part * 16, park);
        }
        const float2 mapv[VEC] = {make_float2(Am.x, H.x), make_float2(Am.y, H.y)};
        mbar_arrive(&empty[s]);  // the stage is read: the producer may refill it
#pragma unroll
        for (int v = 0; v < VEC; ++v) maps[(m * NW + warp) * CHW + lane * VEC + v] = mapv[v];
        mbar_arrive(&maps_ready[m]);
      }
    }
    tmem_wait_st();
    tmem_fence_before_sync();
  }
  __syncthreads();  // every role is done with the block's TMEM
  if (warp == 0) {
    tmem_fence_after_sync();
    __syncwarp();
    tmem_dealloc(*tslot, kChainTmemCols);
  }
}

}  // namespace blr
