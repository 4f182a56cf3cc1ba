// Chained single-pass backward scan: the BD-LRU backward for the problems the
// chained forward serves (few chains, long bfloat16 sequences), reading every
// input from HBM once and writing every output once.
//
// With g_t the total derivative with respect to h_t and w_t = alpha_t g_t the
// adjoint passed to step t - 1, the reverse recurrence g_t = dh_t + w_{t+1}
// (w_L = dh_last) is again a first-order linear scan (Sec. 3.3's operator,
// run from the end): over a run of steps, w leaving its left end is an affine
// map w -> A w + W of the w entering its right end, A the product of the run's
// alphas. Tiles are the forward's kChainTile steps of one chain, numbered
// time-major from the END of the sequence, so that a tile only ever waits on
// tiles of smaller number (those to its right). The block's warps have fixed
// roles:
//   producers (2 warps): one loads tile n's dh and rho into ring A; the other,
//      a little before pass C needs it, tile n's x, rho and iota into ring C
//      (rho is by then in L2), and once pass C has written the tile's outputs
//      over them, sends those out by TMA store before refilling the stage.
//      The first also writes each tile's decay constants and coordinates into
//      a small ring of their own, so that the compute warps divide no tile
//      index;
//   compute (kCbWarps warps, a slice of kCbSlice steps each, which starts at
//      one of the forward's kept states): pass A of tile n evaluates the alphas
//      of its slice and folds the reverse recurrence from a zero carry, last
//      step first (gl_t, and sm_t = the product of the alphas after step t
//      within the slice minus one, so that g_t = gl_t + (1 + sm_t) w_in),
//      parks both in TMEM (16 columns at a time as the fold advances) and
//      publishes the slice's map. Pass C of tile n - kCbLag, once its scanner
//      has found the adjoint entering its slice: starting from the forward's
//      kept state it re-runs the slice forward in time, recomputing each
//      step's gates once, h_{t-1}, g_t and every output (dx, d rho, d iota and
//      the d Lambda terms) in one sweep, writing the outputs over the step's
//      consumed inputs in the ring C stage;
//   scanners (kCbScanners warps, tiles in turn): compose the slice maps into
//      the tile's, chain it to the tiles after it by the decoupled look-back of
//      the forward, publish the adjoint leaving the tile, and hand every slice
//      the adjoint entering it.
// The gradient formulas are those of the serial backward kernels (the chain
// rule of Sec. 3.2's definitions).
#pragma once

#include "blr_chain.cuh"

namespace blr {

constexpr int kCbWarps = 16;                   // compute warps
constexpr int kCbSlice = 8;                    // steps a warp takes of a tile
constexpr int kCbStagesA = 2;                  // ring A stages (dh, rho)
constexpr int kCbStagesC = 2;                  // ring C stages (x, rho, iota)
constexpr int kCbLag = 3;                      // pass C runs this many tiles behind pass A
constexpr int kCbSlots = kCbLag + 1;           // slice-map, adjoint and TMEM slots
constexpr int kCbScanners = 2;
constexpr int kCbThreads = (kCbWarps + kCbScanners + 2) * 32;
constexpr uint32_t kCbTmemCols = 512;
// Registers per thread, as kChainMaxRegs.
constexpr int kCbMaxRegs = (16384 / (((kCbThreads / 32 + 3) / 4) * 32)) / 8 * 8;
// Tiles' decay constants and coordinates, a ring indexed by tile: the ring-A
// producer writes tile i's once pass A of tile i - kCbStagesA has freed its
// stage, and pass C of tile i - kCbStagesA - kCbLag + 1 may still be to run.
constexpr int kCbRates = 8;
static_assert(kCbRates > kCbLag + kCbStagesA, "a tile's decay constants outlive its pass C");
static_assert(kCbWarps * kCbSlice == kChainTile, "the backward tiles are the forward's");

struct ChainBwdArgs {
  CUtensorMap tm_dh;
  CUtensorMap tm_x;
  CUtensorMap tm_r;
  CUtensorMap tm_i;
  CUtensorMap tm_dx;  // the outputs, stored from ring C by TMA
  CUtensorMap tm_dr;
  CUtensorMap tm_di;
  Plan p;
  const float* dh_last;
  const float* lambda;
  const float* h0;
  float* dlambda;
  float* dh0;
  unsigned char* ws;
};

// Shared memory from a 128-byte aligned base, every region 16-byte aligned.
template <typename T, int VEC>
struct ChainBwdSmem {
  static constexpr int CHW = 32 * VEC;
  static constexpr uint32_t BOX = kChainTile * CHW * sizeof(T);
  static constexpr size_t up(size_t v) { return (v + 15) / 16 * 16; }
  static constexpr size_t ringA = 0;                                         // [SA][dh, rho]
  static constexpr size_t ringC = ringA + (size_t)kCbStagesA * 2 * BOX;      // [SC][x, rho, iota]
  static constexpr size_t rates = ringC + (size_t)kCbStagesC * 3 * BOX;     // float2 [kCbRates][CHW]
  static constexpr size_t poly = up(rates + (size_t)kCbRates * CHW * sizeof(float2));  // int [kCbRates]
  static constexpr size_t tmeta = up(poly + (size_t)kCbRates * sizeof(int));  // int4 [kCbRates]
  static constexpr size_t maps = up(tmeta + (size_t)kCbRates * sizeof(int4));  // float2 [MS][W][CHW]
  static constexpr size_t tmem = up(maps + (size_t)kCbSlots * kCbWarps * CHW * sizeof(float2));
  static constexpr size_t bars = up(tmem + sizeof(uint32_t));
  static constexpr size_t end =
      bars + (size_t)(2 * kCbStagesA + 2 * kCbStagesC + 2 * kCbSlots) * sizeof(uint64_t);
  static constexpr size_t bytes = end + 128;
  static_assert(ringC % 128 == 0 && rates % 16 == 0 && maps % 16 == 0 && bars % 16 == 0, "");
};

// Pass A for a bfloat16 lane (two channels as one float2), one part of its
// slice: rows QS-1 .. 0 at lb (rows from `valid` on lie past the sequence and
// act as the identity: alpha = 1, dh = 0), continuing the fold (w, m) of the
// slice's later rows (zero at the slice's end). Row r's g for a zero adjoint
// entering the slice and sm = the product of the alphas of the slice's rows
// after r minus one go to park[4r, 4r + 4) as (g.x, g.y, sm.x, sm.y); on
// return (m, w) is the map of the rows folded so far.
template <bool POLY>
__device__ __forceinline__ void chain_bwd_fold_part_bf16x2(const unsigned char* lb, float2 kh,
                                                           int valid, float2& w, float2& m,
                                                           float (&park)[16]) {
  constexpr int QS = 4;
  constexpr uint32_t ROWB = 128;
  constexpr uint32_t BOX = kChainTile * ROWB;
#pragma unroll
  for (int r = QS - 1; r >= 0; --r) {
    float2 dh = bf2_unpack(*reinterpret_cast<const uint32_t*>(lb + r * ROWB));
    const float2 hr = bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + BOX + r * ROWB), kBf2Half);
    float2 e = expm1_neg2<POLY>(__ffma2_rn(kh, tanh2(hr), kh));
    if (r >= valid) {
      e = f2(0.0f);
      dh = f2(0.0f);
    }
    const float2 g = __fadd2_rn(dh, w);
    park[4 * r] = g.x;
    park[4 * r + 1] = g.y;
    park[4 * r + 2] = m.x;
    park[4 * r + 3] = m.y;
    const float2 alpha = __fadd2_rn(f2(1.0f), e);
    m = __ffma2_rn(alpha, m, e);  // alpha (1 + m) - 1
    w = __fmul2_rn(alpha, g);
  }
}

// Pass C for a bfloat16 lane (two channels as one float2), one part of its
// slice: rows 0 .. QS-1 at lb forward in time from h before them (hp, updated
// to h after them), each step's gates evaluated once (as the serial kernels
// evaluate them) for the state, g_t = gl_t + (1 + sm_t) w_in and the
// gradients, which overwrite the row's x, rho and iota in the stage (dx,
// d rho, d iota: the TMA store clips rows past the sequence); rows from `rows`
// on are not summed. pr holds (gl, sm) of row r at [4r, 4r + 4); kq = k/4 and
// nkq = -k/4 per channel. Adds the d Lambda terms dl_t r_t to dlr; dh0, if not
// NULL, receives alpha_0 g_0 of the part's first row (the sequence's first).
template <bool POLY>
__device__ __forceinline__ void chain_bwd_rows(unsigned char* lb, const uint32_t (&pr)[16], float2 win,
                                               float2 kq, float2 nkq, float2 kh, int rows, float2& hp,
                                               float* dh0, float2& dlr) {
  constexpr int QS = 4;
  constexpr uint32_t ROWB = 128;
  constexpr uint32_t BOX = kChainTile * ROWB;
#pragma unroll
  for (int r = 0; r < QS; ++r) {
    const float2 gl = make_float2(__uint_as_float(pr[4 * r]), __uint_as_float(pr[4 * r + 1]));
    const float2 smr = make_float2(__uint_as_float(pr[4 * r + 2]), __uint_as_float(pr[4 * r + 3]));
    const float2 nhx = bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + r * ROWB), kBf2NegHalf);
    const float2 thr = tanh2(bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + BOX + r * ROWB), kBf2Half));
    const float2 thi = tanh2(bf2_scaled(*reinterpret_cast<const uint32_t*>(lb + 2 * BOX + r * ROWB), kBf2Half));
    const float2 e = expm1_neg2<POLY>(__ffma2_rn(kh, thr, kh));
    const float2 alpha = __fadd2_rn(f2(1.0f), e);
    const float2 m2 = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // -(1 - alpha^2)
    const float2 rs = make_float2(rsqrt_approx(fmaxf(-m2.x, 1e-30f)), rsqrt_approx(fmaxf(-m2.y, 1e-30f)));
    const float2 nq = __fmul2_rn(m2, rs);                // -sqrt(1 - alpha^2)
    const float2 nix = __ffma2_rn(nhx, thi, nhx);        // -i x
    const float2 g = map_apply2(smr, win, gl);           // g_t = gl_t + (1 + sm_t) w_in
    const float2 w = __fmul2_rn(alpha, g);
    const float2 gnq = __fmul2_rn(g, nq);                // -g sqrt(1 - alpha^2)
    const float2 ni = __ffma2_rn(f2(-0.5f), thi, f2(-0.5f));  // -i
    const float2 omi = __ffma2_rn(f2(-0.5f), thi, f2(0.5f));  // 1 - i
    // dx = g sqrt(1 - alpha^2) i; d iota = g u (1 - i);
    // d l = alpha g (h_{t-1} - alpha i x / sqrt(1 - alpha^2)); d rho = d l k r (1 - r),
    // r (1 - r) = (1 - tanh(rho/2)^2) / 4
    const float2 ox = __fmul2_rn(gnq, ni);
    const float2 oi = __fmul2_rn(__fmul2_rn(gnq, nix), omi);
    const float2 dl = __fmul2_rn(w, __ffma2_rn(__fmul2_rn(alpha, rs), nix, hp));
    const float2 orho = __fmul2_rn(dl, __ffma2_rn(nkq, __fmul2_rn(thr, thr), kq));
    hp = __ffma2_rn(alpha, hp, __fmul2_rn(nq, nix));  // alpha h + sqrt(1 - alpha^2) i x
    *reinterpret_cast<uint32_t*>(lb + r * ROWB) = bf2_pack(ox);
    *reinterpret_cast<uint32_t*>(lb + BOX + r * ROWB) = bf2_pack(orho);
    *reinterpret_cast<uint32_t*>(lb + 2 * BOX + r * ROWB) = bf2_pack(oi);
    if (r < rows) {
      dlr = __ffma2_rn(dl, __ffma2_rn(f2(0.5f), thr, f2(0.5f)), dlr);  // += d l r
      if (dh0 != nullptr && r == 0) {  // the sequence's first step: dh0 = alpha_0 g_0
        dh0[0] = w.x;
        dh0[1] = w.y;
      }
    }
  }
}

// ------------------------------------------------------------------- kernel

template <typename T, class M, int VEC, int RB>
__global__ void __maxnreg__(kCbMaxRegs) chain_bwd_kernel(const __grid_constant__ ChainBwdArgs a) {
  using IO = Io<T, VEC>;
  using G = typename GatePolicy<M>::type;
  using SM = ChainBwdSmem<T, VEC>;
  constexpr int CHW = 32 * VEC;
  constexpr int SA = kCbStagesA, SC = kCbStagesC, NW = kCbWarps, TS = kCbSlice, MS = kCbSlots;
  constexpr int LAG = kCbLag;
  constexpr uint32_t ROWB = CHW * sizeof(T);
  constexpr uint32_t BOX = SM::BOX;
  static_assert(VEC == 2 && G::kHalfInputs, "the chained backward is the bfloat16 path");
  static_assert(TS % RB == 0 && kChainTile % RB == 0, "every slice starts at a kept state");
  static_assert(TS == 8, "a slice is two parts of 4 rows, 16 TMEM columns each");
  static_assert(NW % 4 == 0 && (NW / 4) * 32 * MS <= kCbTmemCols, "TMEM slots");
  const Plan& p = a.p;
  extern __shared__ unsigned char chain_smem[];
  unsigned char* base = align128(chain_smem);
  float2* rates = reinterpret_cast<float2*>(base + SM::rates);  // [kCbRates][CHW]: (k, k/2)
  int* polys = reinterpret_cast<int*>(base + SM::poly);
  int4* tmeta = reinterpret_cast<int4*>(base + SM::tmeta);  // [kCbRates]: tile coordinates
  float2* maps = reinterpret_cast<float2*>(base + SM::maps);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(base + SM::tmem);
  uint64_t* fullA = reinterpret_cast<uint64_t*>(base + SM::bars);
  uint64_t* emptyA = fullA + SA;
  uint64_t* fullC = emptyA + SA;
  uint64_t* writtenC = fullC + SC;  // a ring C stage holds its tile's outputs
  uint64_t* maps_ready = writtenC + SC;
  uint64_t* carry_ready = maps_ready + MS;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(a.ws + p.off_bhdr);
  uint32_t* err = &fh->err;
  {
    __shared__ int s_ok;
    if (threadIdx.x == 0) {
      s_ok = __ldcg(&fh->tag) == seg_tag(p.tag) && __ldcg(&fh->complete) == 1u;
      if (!s_ok) atomicOr(&fh->err, kErrWorkspace);
    }
    __syncthreads();
    if (!s_ok) return;  // no forward states for this problem: write nothing
  }
  const int64_t C = p.n_chain;
  const int64_t n_g = (p.D + CHW - 1) / CHW;
  const int64_t BD = p.B * p.D;
  const int64_t n_tc = p.n_tc;
  const int64_t n_tiles = n_tc * C;
  const int64_t G_ = gridDim.x;
  const int64_t n_my = blockIdx.x < n_tiles ? (n_tiles - blockIdx.x + G_ - 1) / G_ : 0;

  if (warp == 0) {
    __syncwarp();
    tmem_alloc(tslot, kCbTmemCols);
    tmem_fence_before_sync();
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < SA; ++s) {
      mbar_init(&fullA[s], 1);
      mbar_init(&emptyA[s], NW * 32);
    }
    for (int s = 0; s < SC; ++s) {
      mbar_init(&fullC[s], 1);
      mbar_init(&writtenC[s], NW * 32);
    }
    for (int m = 0; m < MS; ++m) {
      mbar_init(&maps_ready[m], NW * 32);
      mbar_init(&carry_ready[m], 32);
    }
    fence_mbar_init();
  }
  __syncthreads();  // the roles part here and meet again at the end

  // Tile n of this block: (time block, batch row, channel group), time blocks
  // counted from the end of the sequence.
  const uint32_t C32 = (uint32_t)C, ng32 = (uint32_t)n_g;
  auto coord = [&](int64_t n) {
    const uint32_t tile = (uint32_t)(blockIdx.x + n * G_);
    const uint32_t q = tile / C32, chain = tile - q * C32;
    const uint32_t b = chain / ng32;
    return make_int4((int)(n_tc - 1 - q), (int)b, (int)(chain - b * ng32), 0);
  };

  if (warp == NW + kCbScanners) {
    // ---------------------------------------------------------- producer A
    // Tile i's dh and rho into ring A, with its decay constants (k, k/2) and
    // POLY flag in the rates ring, once the stage is free. The constants of
    // tile i + 1 are evaluated (their Lambda loads in flight) while the stage
    // for tile i is awaited.
    float k[VEC], kh[VEC], nk[VEC], nkh[VEC];
    int npoly = 0;
    auto prep = [&](int64_t i) {
      const int4 c = coord(i);
      const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
      npoly = seq_rates<VEC>(a.lambda, p.c, d0, d0 < p.D, nk, nkh) ? 1 : 0;
    };
    if (n_my > 0) prep(0);
    for (int64_t i = 0; i < n_my; ++i) {
      const int s = (int)(i % SA);
      const int rr = (int)(i % kCbRates);
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        k[v] = nk[v];
        kh[v] = nkh[v];
      }
      const int poly = npoly;
      if (i + 1 < n_my) prep(i + 1);
      if (i >= SA) mbar_wait(&emptyA[s], (uint32_t)(i / SA - 1) & 1u, err);
#pragma unroll
      for (int v = 0; v < VEC; ++v) rates[rr * CHW + lane * VEC + v] = make_float2(k[v], kh[v]);
      const int4 c = coord(i);
      if (lane == 0) {
        polys[rr] = poly;
        tmeta[rr] = c;
      }
      __syncwarp();
      if (lane == 0) {  // the arrival releases the constants with the stage
        unsigned char* dst = base + SM::ringA + (size_t)s * 2 * BOX;
        const int t = c.x * kChainTile, cd = c.z * CHW, cb = c.y;
        mbar_arrive_expect_tx(&fullA[s], 2 * BOX);
        tma_load_3d(dst, &a.tm_dh, &fullA[s], cd, t, cb);
        tma_load_3d(dst + BOX, &a.tm_r, &fullA[s], cd, t, cb);
      }
    }
  } else if (warp == NW + kCbScanners + 1) {
    // ---------------------------------------------------------- producer C
    // Step q: once pass C of tile q - SC has written its outputs over its
    // stage, sends them out (dx, d rho, d iota: three TMA stores, clipped to
    // the tensors) and, as soon as the stores have read the stage, loads tile
    // q's x, rho and iota into it.
    if (lane == 0) {
      for (int64_t q = 0; q < n_my + SC; ++q) {
        const int s = (int)(q % SC);
        unsigned char* stg = base + SM::ringC + (size_t)s * 3 * BOX;
        if (q >= SC) {
          const int64_t j = q - SC;
          mbar_wait(&writtenC[s], (uint32_t)(j / SC) & 1u, err);
          const int4 c = coord(j);
          const int t = c.x * kChainTile, cd = c.z * CHW, cb = c.y;
          tma_store_3d(&a.tm_dx, stg, cd, t, cb);
          tma_store_3d(&a.tm_dr, stg + BOX, cd, t, cb);
          tma_store_3d(&a.tm_di, stg + 2 * BOX, cd, t, cb);
          bulk_commit();
          bulk_wait_read<0>();  // the stage is free once the stores have read it
        }
        if (q < n_my) {
          const int4 c = coord(q);
          const int t = c.x * kChainTile, cd = c.z * CHW, cb = c.y;
          mbar_arrive_expect_tx(&fullC[s], 3 * BOX);
          tma_load_3d(stg, &a.tm_x, &fullC[s], cd, t, cb);
          tma_load_3d(stg + BOX, &a.tm_r, &fullC[s], cd, t, cb);
          tma_load_3d(stg + 2 * BOX, &a.tm_i, &fullC[s], cd, t, cb);
        }
      }
      bulk_wait_all();  // every store complete before the block ends
    }
    __syncwarp();
  } else if (warp >= NW) {
    // ---------------------------------------------------------- scanners
    unsigned long long* agg = reinterpret_cast<unsigned long long*>(a.ws + p.off_cagg);
    uint32_t* inc = reinterpret_cast<uint32_t*>(a.ws + p.off_cinc);
    for (int64_t n = warp - NW; n < n_my; n += kCbScanners) {
      const int m = (int)(n % MS);
      const int4 c = coord(n);
      const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
      const bool ch_ok = d0 < p.D;
      mbar_wait(&maps_ready[m], (uint32_t)(n / MS) & 1u, err);
      // the tile's map: its slices from the last to the first
      float TM[VEC], TU[VEC], ws[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        TM[v] = 0.0f;
        TU[v] = 0.0f;
#pragma unroll
        for (int w = NW - 1; w >= 0; --w) {
          const float2 e = maps[(m * NW + w) * CHW + lane * VEC + v];
          TU[v] = map_apply(e.x, TU[v], e.y);
          TM[v] = m_compose(TM[v], e.x);
        }
        ws[v] = 0.0f;
      }
      if (ch_ok) {
        const int64_t ch0 = (int64_t)c.y * p.D + d0;
        const int64_t rec = (int64_t)c.x * BD + ch0;
        if (c.x == n_tc - 1) {  // the sequence's last time block: the adjoint entering is dh_last
          if (a.dh_last != nullptr) {
#pragma unroll
            for (int v = 0; v < VEC; ++v) ws[v] = a.dh_last[ch0 + v];
          }
        } else {
#pragma unroll
          for (int v = 0; v < VEC; ++v) st_record(&agg[rec + v], pack_agg(TM[v], TU[v]));
          // predecessors: time blocks c.x + 1, c.x + 2, ..., n_tc - 1
          const int64_t near = rec + BD, nprev = n_tc - 1 - c.x;
          ChainWindow win[VEC];
#pragma unroll
          for (int v = 0; v < VEC; ++v) chain_window_load(agg + near + v, inc + near + v, BD, 0, nprev, win[v]);
#pragma unroll
          for (int v = 0; v < VEC; ++v) ws[v] = chain_walk(agg + near + v, inc + near + v, BD, nprev, err, win[v]);
        }
#pragma unroll
        for (int v = 0; v < VEC; ++v) st_record(&inc[rec + v], __float_as_uint(map_apply(TM[v], ws[v], TU[v])));
      }
      // the adjoint entering every slice, written over the slice's map
#pragma unroll
      for (int w = NW - 1; w >= 0; --w) {
#pragma unroll
        for (int v = 0; v < VEC; ++v) {
          float2* e = &maps[(m * NW + w) * CHW + lane * VEC + v];
          const float2 mw = *e;
          e->x = ws[v];
          ws[v] = map_apply(mw.x, ws[v], mw.y);
        }
      }
      mbar_arrive(&carry_ready[m]);
    }
  } else {
    // ---------------------------------------------------------- compute
    // Pass A of tile n parks (gl, sm) of the slice's rows in TMEM slot n % MS
    // of this warp's lanes (32 columns: rows 0-3, then rows 4-7); pass C of
    // tile n - LAG takes them back. Each iteration runs C first, so that A's
    // park stores have a whole iteration to complete before the next A waits
    // for them.
    tmem_fence_after_sync();
    constexpr uint32_t kWarpCols = 32;
    constexpr uint32_t kSlotCols = (NW / 4) * kWarpCols;
    constexpr int QS = 4;
    const uint32_t tq = *tslot + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(warp >> 2) * kWarpCols;
    const float* kept = reinterpret_cast<const float*>(a.ws + p.off_skept);
    double* acc = reinterpret_cast<double*>(a.ws + p.off_dlam);
    const uint32_t loff = warp * TS * ROWB + lane * VEC * sizeof(T);  // this lane's first row
    const uint32_t nmy = (uint32_t)n_my;
    for (uint32_t n = 0; n < nmy + LAG; ++n) {
      if (n >= LAG) {
        // ---- C: tile n - LAG, forward in time from the forward's kept state
        const uint32_t q = n - LAG;
        const uint32_t m = q % MS, sc = q % SC;
        const int4 c = tmeta[q % kCbRates];
        const int64_t d0 = (int64_t)c.z * CHW + lane * VEC;
        const int64_t t0 = (int64_t)c.x * kChainTile + warp * TS;
        const int64_t row0 = (int64_t)c.y * p.D + d0;  // (batch row, channel) offset of a state
        const bool ch_ok = d0 < p.D;
        // h before the slice: the kept state after step t0 - 1 (h0, or zero, for t0 = 0)
        float2 hp = make_float2(0.0f, 0.0f);
        if (ch_ok && t0 < p.L) {  // kept state t0 / RB - 1 exists for 0 < t0 < L
          if (t0 > 0)
            hp = __ldcg(reinterpret_cast<const float2*>(kept + (t0 / RB - 1) * BD + row0));
          else if (a.h0 != nullptr)
            hp = make_float2(a.h0[row0], a.h0[row0 + 1]);
        }
        uint32_t pr[16];
        __syncwarp();  // tcgen05 accesses are warp-collective
        tmem_ld16_start(tq + m * kSlotCols, pr);
        mbar_wait(&carry_ready[m], (q / MS) & 1u, err);
        mbar_wait(&fullC[sc], (q / SC) & 1u, err);
        const float2 win = make_float2(maps[(m * NW + warp) * CHW + lane * VEC].x,
                                       maps[(m * NW + warp) * CHW + lane * VEC + 1].x);
        const uint32_t rq = q % kCbRates;
        const float2 r0 = rates[rq * CHW + lane * VEC], r1 = rates[rq * CHW + lane * VEC + 1];
        const float2 kq = make_float2(0.25f * r0.x, 0.25f * r1.x), nkq = make_float2(-kq.x, -kq.y);
        const float2 kh = make_float2(r0.y, r1.y);
        const bool poly = polys[rq] != 0;
        __syncwarp();
        tmem_ld_wait(pr);
        unsigned char* lb = base + SM::ringC + sc * (3 * BOX) + loff;
        const int rows = !ch_ok || t0 >= p.L ? 0 : (p.L - t0 < TS ? (int)(p.L - t0) : TS);
        const int rows0 = rows < QS ? rows : QS, rows1 = rows - rows0;
        float* pd0 = (t0 == 0 && ch_ok) ? a.dh0 : nullptr;
        if (pd0 != nullptr) pd0 += row0;
        float2 dlr = make_float2(0.0f, 0.0f);
        if (poly)
          chain_bwd_rows<true>(lb, pr, win, kq, nkq, kh, rows0, hp, pd0, dlr);
        else
          chain_bwd_rows<false>(lb, pr, win, kq, nkq, kh, rows0, hp, pd0, dlr);
        __syncwarp();
        tmem_ld16_start(tq + m * kSlotCols + 16, pr);
        tmem_ld_wait(pr);
        if (poly)
          chain_bwd_rows<true>(lb + QS * ROWB, pr, win, kq, nkq, kh, rows1, hp, nullptr, dlr);
        else
          chain_bwd_rows<false>(lb + QS * ROWB, pr, win, kq, nkq, kh, rows1, hp, nullptr, dlr);
        fence_proxy_async_smem();  // this thread's outputs in the stage, visible to the TMA stores
        mbar_arrive(&writtenC[sc]);
        // d Lambda: this slice's terms into the float64 partial sums (reductions
        // without a result, striped over batch rows)
        if (rows > 0) {
          double* ad = acc + (c.y % kStripes) * p.D + d0;
          atomicAdd(ad, (double)dlr.x);
          atomicAdd(ad + 1, (double)dlr.y);
        }
      }
      if (n < nmy) {
        // ---- A: tile n's reverse fold from a zero adjoint, rows 7-4 then
        // 3-0, each part parked as soon as it is folded; the stage is free
        // afterwards
        const uint32_t s = n % SA, m = n % MS;
        tmem_wait_st();  // the previous tile's park stores, before a later load of their slot
        mbar_wait(&fullA[s], (n / SA) & 1u, err);
        const int4 c = tmeta[n % kCbRates];
        const int64_t t0 = (int64_t)c.x * kChainTile + warp * TS;
        const int valid = t0 >= p.L ? 0 : (p.L - t0 < TS ? (int)(p.L - t0) : TS);
        const int valid1 = valid > QS ? valid - QS : 0, valid0 = valid < QS ? valid : QS;
        const unsigned char* lb = base + SM::ringA + s * (2 * BOX) + loff;
        const uint32_t rn = n % kCbRates;
        const float2 kh = make_float2(rates[rn * CHW + lane * VEC].y, rates[rn * CHW + lane * VEC + 1].y);
        const bool poly = polys[rn] != 0;
        float2 w = make_float2(0.0f, 0.0f), mm = make_float2(0.0f, 0.0f);
        float park[16];
        if (poly)
          chain_bwd_fold_part_bf16x2<true>(lb + QS * ROWB, kh, valid1, w, mm, park);
        else
          chain_bwd_fold_part_bf16x2<false>(lb + QS * ROWB, kh, valid1, w, mm, park);
        __syncwarp();
        tmem_st16(tq + m * kSlotCols + 16, park);
        if (poly)
          chain_bwd_fold_part_bf16x2<true>(lb, kh, valid0, w, mm, park);
        else
          chain_bwd_fold_part_bf16x2<false>(lb, kh, valid0, w, mm, park);
        __syncwarp();
        tmem_st16(tq + m * kSlotCols, park);
        mbar_arrive(&emptyA[s]);
        maps[(m * NW + warp) * CHW + lane * VEC] = make_float2(mm.x, w.x);
        maps[(m * NW + warp) * CHW + lane * VEC + 1] = make_float2(mm.y, w.y);
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
    tmem_dealloc(*tslot, kCbTmemCols);
  }
  // The last block out turns the partial sums into d Lambda and clears them
  // (and the exit counter) for the next backward.
  __shared__ int s_last;
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&bh->exited, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    double* acc = reinterpret_cast<double*>(a.ws + p.off_dlam);
    for (int64_t d = threadIdx.x; d < p.D; d += blockDim.x) {
      double sum = 0.0;
      for (int s2 = 0; s2 < kStripes; ++s2) {
        sum += __ldcg(&acc[s2 * p.D + d]);
        acc[s2 * p.D + d] = 0.0;
      }
      const double lam = (double)a.lambda[d];
      const double sig = 1.0 / (1.0 + exp(-lam));  // d softplus / d Lambda
      a.dlambda[d] = (float)(-(double)p.c * sig * sum);
    }
    if (threadIdx.x == 0) bh->exited = 0u;
  }
}

}  // namespace blr
