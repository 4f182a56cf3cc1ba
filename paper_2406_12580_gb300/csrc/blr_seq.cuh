// Serial scan kernels: the BD-LRU scan when a problem has enough independent
// (batch row, channel group) chains to fill the GPU by itself.
//
// One warp (one thread block) owns CHW = 32 * VEC consecutive channels of one
// batch row, a 128-byte row segment, and walks the whole sequence: each lane
// runs the recurrence h_t = alpha_t h_{t-1} + beta_t x_t of Sec. 3.2 serially
// for its VEC channels, one multiply-add per element, with the state in
// registers. There is no cross-lane or cross-block combine and no second pass.
//
// Data movement is TMA both ways. The inputs stream through a ring of
// shared-memory stages, one box of R rows per tensor; each lane writes
// its outputs over its own, already consumed, inputs in the stage, and one TMA
// store per output tensor sends the stage's outputs to global memory, clipped
// to the tensor's extent (sequence and channel tails need no masking). A stage
// is refilled at the start of the next iteration, once its store has read it,
// so two stages already double-buffer.
//
// The forward also keeps the state after every RB steps, which the backward
// uses as its starting points: the backward walks the sequence from the end in
// sub-blocks of RB steps, recomputes the sub-block's gates and states forward
// from the kept state (holding E = alpha - 1, 1 / sqrt(1 - alpha^2) and
// h_{t-1} per element in registers; bfloat16 lanes: alpha, sqrt(1 - alpha^2)
// and the d l factor), then runs the reverse recurrence
// g_t = dh_t + alpha_{t+1} g_{t+1} through it, writing dx, d rho and d iota and
// accumulating d Lambda. bfloat16 lanes carry their two channels as packed
// float pairs (paired multiply-adds).
//
// The forward's first block also restarts the workspace bookkeeping (error
// word, problem tag, the backward's exit counter and d Lambda partial sums), so
// no preparation kernel runs before either scan.
#pragma once

#include "blr_kernels.cuh"

namespace blr {

constexpr int kSeqMaxStages = 8;   // ring stages per warp
// Rings of at least this many stages may refill a consumed stage after the
// next stage's arithmetic rather than before it (the kernels' LATE form;
// measured on GB300: float32 rings of 4-8 stages up to 5 % faster that way,
// bfloat16 rings of 2-3 stages 3-7 % slower, so bfloat16 keeps the early
// form).
constexpr int kSeqLateRefillStages = 4;

// Tensor maps: (channels, time, batch) views with boxes of 32 * VEC channels x
// R steps x 1 row. gate_logits is seen as two views of D channels each
// (rho: columns [0, D), iota: columns [D, 2D)), so that boxes clip at D.
struct SeqFwdArgs {
  CUtensorMap tm_x;
  CUtensorMap tm_r;
  CUtensorMap tm_i;
  CUtensorMap tm_h;  // h, or y = h SiLU(z) when gated; unused when NULL
  CUtensorMap tm_z;  // gated: z, the merge gate's input
  Plan p;
  const int32_t* lengths;  // NULL, or row b's sequence is its last lengths[b] steps
  const float* lambda;
  const float* h0;
  float* h_last;
  unsigned char* ws;
  int stages;
  int write_h;
};

struct SeqBwdArgs {
  CUtensorMap tm_dh;
  CUtensorMap tm_x;
  CUtensorMap tm_r;
  CUtensorMap tm_i;
  CUtensorMap tm_dx;
  CUtensorMap tm_dr;
  CUtensorMap tm_di;
  CUtensorMap tm_z;   // gated: z
  CUtensorMap tm_dz;  // gated: dz
  Plan p;
  const int32_t* lengths;  // as SeqFwdArgs
  const float* dh_last;
  const float* lambda;
  const float* h0;
  float* dlambda;
  float* dh0;
  unsigned char* ws;
  int stages;
};

__device__ __forceinline__ unsigned char* align128(unsigned char* p) {
  const uint32_t a = smem_addr(p);
  return p + (((a + 127u) & ~127u) - a);
}

// Dynamic shared memory of a serial kernel: `stages` stages of NB boxes, one
// mbarrier per stage, and slack for the 128-byte alignment of the boxes.
template <typename T, int VEC, int R>
__host__ __device__ constexpr uint32_t seq_box_bytes() {
  return (uint32_t)(R * 32 * VEC * sizeof(T));
}
template <typename T, int VEC, int R>
inline size_t seq_smem_bytes(int stages, int nb) {
  return (size_t)stages * nb * seq_box_bytes<T, VEC, R>() + (size_t)stages * sizeof(uint64_t) + 128;
}

// Per-lane channel constants: k = -c softplus(Lambda), kh = k / 2, and whether
// every channel of the warp keeps l = k r inside the series' range.
template <int VEC>
__device__ __forceinline__ bool seq_rates(const float* lambda, float c, int64_t d0, bool ch_ok,
                                          float (&k)[VEC], float (&kh)[VEC]) {
  bool poly = true;
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    k[v] = ch_ok ? decay_rate(c, lambda[d0 + v]) : 0.0f;
    kh[v] = 0.5f * k[v];
    poly = poly && k[v] >= -kExpm1Series;
  }
  return __all_sync(kFull, poly);
}

// The ring: stage i holds NB boxes, then the S mbarriers. Block-uniform
// bookkeeping of which stage holds which box and when it may be refilled.
template <int NB, uint32_t BOX>
struct SeqRing {
  unsigned char* base;
  uint64_t* bars;
  int S;
  __device__ __forceinline__ unsigned char* stage(int st) const { return base + (size_t)st * NB * BOX; }
};

// Kernel modes: the plain scan, rows with lengths, or chains cut into time
// segments (the segmented serial kernels).
constexpr int kSeqPlain = 0, kSeqVarlen = 1, kSeqSeg = 2;

// The problem tag a segmented forward leaves in the workspace: distinct from
// the other kernels' (its kept states and maps live elsewhere), so that a
// segmented backward refuses a workspace that another forward filled.
__host__ __device__ constexpr uint32_t seg_tag(uint32_t tag) { return tag ^ 0x80000000u; }

// Restarts the workspace bookkeeping for a forward (one block, one warp):
// clears the error word, the backward's exit counter and the d Lambda partial
// sums, and tags the workspace with the problem.
__device__ __forceinline__ void seq_reset_workspace(unsigned char* ws, const Plan& p, uint32_t tag,
                                                    int lane) {
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(ws + p.off_bhdr);
  double* acc = reinterpret_cast<double*>(ws + p.off_dlam);
  for (int64_t i = lane; i < (int64_t)kStripes * p.D; i += 32) acc[i] = 0.0;
  if (lane == 0) {
    fh->err = 0u;
    bh->exited = 0u;
    fh->tag = tag;
    fh->complete = 1u;
  }
}

// Segmented kernels. The start state of segment sg: h0 carried through the
// maps h -> A h + U of segments 0 .. sg-1 (`agg` points at this lane's
// channels of segment 0; segments are BD float pairs apart). Loads go out
// eight segments at a time; missing ones are the identity map (1, 0).
constexpr int kSegComposeBatch = 8;
template <int VEC>
__device__ __forceinline__ void seg_carry_in(const float2* agg, int64_t BD, int64_t sg,
                                             float (&hc)[VEC]) {
  constexpr int U = kSegComposeBatch;
  for (int64_t s0 = 0; s0 < sg; s0 += U) {
    float2 m[U][VEC];
#pragma unroll
    for (int u = 0; u < U; ++u) {
#pragma unroll
      for (int v = 0; v < VEC; ++v)
        m[u][v] = s0 + u < sg ? __ldcg(agg + (s0 + u) * BD + v) : make_float2(1.0f, 0.0f);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) hc[v] = fmaf(m[u][v].x, hc[v], m[u][v].y);
    }
  }
}

// The adjoint carry at the end of segment sg: w (dh_last) carried backwards
// through the maps w -> A w + W of segments nseg-1 .. sg+1, where A is the
// segment's product of alphas and W its adjoint scan from a zero carry (one
// float pair (A, W) per lane channel and segment, written by the backward's
// segment reduction).
template <int VEC>
__device__ __forceinline__ void seg_adjoint_in(const float2* maps, int64_t BD, int64_t sg,
                                               int64_t nseg, float (&w)[VEC]) {
  constexpr int U = kSegComposeBatch;
  for (int64_t s0 = nseg - 1; s0 > sg; s0 -= U) {
    float2 m[U][VEC];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t s = s0 - u;
#pragma unroll
      for (int v = 0; v < VEC; ++v) m[u][v] = s > sg ? __ldcg(maps + s * BD + v) : make_float2(1.0f, 0.0f);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) w[v] = fmaf(m[u][v].x, w[v], m[u][v].y);
    }
  }
}

// ------------------------------------------------- packed bfloat16 pairs
//
// A bfloat16 lane's two channels as one float2, so that the multiply-adds of
// both run as one paired instruction (fma/mul/add.rn.f32x2); the
// transcendental units (tanh, rsqrt, sqrt) stay scalar. Every paired operation
// rounds each half exactly as its scalar counterpart would.

constexpr uint32_t kBf2Half = 0x3f003f00u;     // (0.5, 0.5) as bfloat16 pairs
constexpr uint32_t kBf2NegHalf = 0xbf00bf00u;  // (-0.5, -0.5)

__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }
// The pair t as floats.
__device__ __forceinline__ float2 bf2_unpack(uint32_t t) {
  return make_float2(__uint_as_float(t << 16), __uint_as_float(t & 0xffff0000u));
}
// The pair t times s2 (a bfloat16 pair of +-0.5: exact, a sign and exponent
// change), as floats.
__device__ __forceinline__ float2 bf2_scaled(uint32_t t, uint32_t s2) {
  uint32_t u;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(u) : "r"(t), "r"(s2));
  return bf2_unpack(u);
}
__device__ __forceinline__ uint32_t bf2_pack(float2 v) { return pack_bf16x2(v.x, v.y); }
// A shared-memory word read afresh where it is used, never kept in a register
// from an earlier read of the same word (the backward re-reads a step's inputs
// instead of holding them, and their gates, across a sub-block).
__device__ __forceinline__ uint32_t lds_again(const unsigned char* p) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(smem_addr(p)));
  return v;
}
__device__ __forceinline__ float2 tanh2(float2 a) {
  return make_float2(tanh_approx(a.x), tanh_approx(a.y));
}
// e^l - 1 for l <= 0 (GatesFast: the degree-4 series, ex2 beyond its range
// unless POLY), as expm1_neg<4, POLY> on each half.
template <bool POLY>
__device__ __forceinline__ float2 expm1_neg2(float2 l) {
  if constexpr (POLY) {
    float2 q = __ffma2_rn(f2(1.0f / 24), l, f2(1.0f / 6));
    q = __ffma2_rn(q, l, f2(0.5f));
    q = __ffma2_rn(q, l, f2(1.0f));
    return __fmul2_rn(q, l);
  } else {
    return make_float2(expm1_neg<4, false>(l.x), expm1_neg<4, false>(l.y));
  }
}

// ------------------------------------------------------------------ forward

// seq_fwd_stage for a bfloat16 lane under GatesFast, without the merge: the
// same arithmetic in the same order, on packed pairs.
template <bool POLY, bool FULL, int R, int RB>
__device__ __forceinline__ void seq_fwd_stage_bf16x2(unsigned char* sb, int rows, float2 kh,
                                                     float2& hc, float* carry, int64_t& cidx,
                                                     int64_t n_carry, int64_t BD, bool ch_ok) {
  constexpr uint32_t ROWB = 128;
  constexpr uint32_t BOX = R * ROWB;
  float2 al[R], uu[R];
#pragma unroll
  for (int s = 0; s < R; ++s) {
    if (FULL || s < rows) {
      const float2 hx = bf2_scaled(*reinterpret_cast<const uint32_t*>(sb + s * ROWB), kBf2Half);
      const float2 hr = bf2_scaled(*reinterpret_cast<const uint32_t*>(sb + BOX + s * ROWB), kBf2Half);
      const float2 hi = bf2_scaled(*reinterpret_cast<const uint32_t*>(sb + 2 * BOX + s * ROWB), kBf2Half);
      const float2 e = expm1_neg2<POLY>(__ffma2_rn(kh, tanh2(hr), kh));  // l = kh tanh(rho/2) + kh
      al[s] = __fadd2_rn(f2(1.0f), e);
      const float2 m2 = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // -(1 - alpha^2)
      const float2 n = make_float2(sqrt_approx(-m2.x), sqrt_approx(-m2.y));
      uu[s] = __fmul2_rn(n, __ffma2_rn(hx, tanh2(hi), hx));  // sqrt(1 - alpha^2) i x
    }
  }
#pragma unroll
  for (int s = 0; s < R; ++s) {
    if (FULL || s < rows) {
      hc = __ffma2_rn(al[s], hc, uu[s]);
      *reinterpret_cast<uint32_t*>(sb + s * ROWB) = bf2_pack(hc);
      if ((s + 1) % RB == 0) {  // a kept state: after step (cidx + 1) RB - 1
        if (cidx < n_carry && ch_ok) *reinterpret_cast<float2*>(carry + cidx * BD) = hc;
        ++cidx;
      }
    }
  }
}

// One stage, rows [0, rows) (all R when FULL). Phase 1 evaluates the
// gates of every row (independent work), phase 2 runs the recurrence and
// writes h over x in the stage (GATED: y = h SiLU(z), the merge of the gated
// recurrent layer, Alg. 1, with z the stage's fourth box). `cidx` is the index
// of the next kept state.
template <class IO, class G, bool POLY, bool FULL, int R, int RB, bool GATED>
__device__ __forceinline__ void seq_fwd_stage(unsigned char* sb, int rows,
                                              const float (&k)[IO::VEC], const float (&kh)[IO::VEC],
                                              float (&hc)[IO::VEC], float* carry, int64_t& cidx,
                                              int64_t n_carry, int64_t BD, bool ch_ok) {
  using Raw = typename IO::Raw;
  constexpr int V = IO::VEC;
  constexpr uint32_t ROWB = 32 * V * sizeof(typename IO::T);
  constexpr uint32_t BOX = R * ROWB;
  float al[R][V], uu[R][V];
#pragma unroll
  for (int s = 0; s < R; ++s) {
    if (FULL || s < rows) {
      float xv[V], rv[V], iv[V];
      if constexpr (G::kHalfInputs) {
        IO::unpack_half(*reinterpret_cast<const Raw*>(sb + s * ROWB), xv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(sb + BOX + s * ROWB), rv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(sb + 2 * BOX + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          const float e = expm1_neg<G::kDeg, POLY>(G::decay_log_half(rv[v], kh[v]));
          al[s][v] = 1.0f + e;
          uu[s][v] = G::sqrt(-e * (e + 2.0f)) * G::gated_x_half(iv[v], xv[v]);
        }
      } else {
        IO::unpack(*reinterpret_cast<const Raw*>(sb + s * ROWB), xv);
        IO::unpack(*reinterpret_cast<const Raw*>(sb + BOX + s * ROWB), rv);
        IO::unpack(*reinterpret_cast<const Raw*>(sb + 2 * BOX + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          const float e = expm1_neg<G::kDeg, POLY>(G::decay_log(rv[v], k[v], kh[v]));
          al[s][v] = 1.0f + e;
          uu[s][v] = G::sqrt(-e * (e + 2.0f)) * (G::sigmoid(iv[v]) * xv[v]);
        }
      }
    }
  }
#pragma unroll
  for (int s = 0; s < R; ++s) {
    if (FULL || s < rows) {
      float out[V];
      // SiLU(z) here rather than with the gates: off the gates' dependency
      // chains, it overlaps the recurrence (measured faster).
      float sz[V];
      if constexpr (GATED) {
        float zv[V];
        if constexpr (G::kHalfInputs)
          IO::unpack_half(*reinterpret_cast<const Raw*>(sb + 3 * BOX + s * ROWB), zv);
        else
          IO::unpack(*reinterpret_cast<const Raw*>(sb + 3 * BOX + s * ROWB), zv);
#pragma unroll
        for (int v = 0; v < V; ++v) sz[v] = G::silu(zv[v]);
      }
#pragma unroll
      for (int v = 0; v < V; ++v) {
        hc[v] = fmaf(al[s][v], hc[v], uu[s][v]);
        if constexpr (GATED)
          out[v] = hc[v] * sz[v];
        else
          out[v] = hc[v];
      }
      IO::store_smem(sb + s * ROWB, out);
      if ((s + 1) % RB == 0) {  // a kept state: after step (cidx + 1) RB - 1
        if (cidx < n_carry && ch_ok) {
#pragma unroll
          for (int v = 0; v < V; ++v) carry[cidx * BD + v] = hc[v];
        }
        ++cidx;
      }
    }
  }
}

// MODE kSeqVarlen: the rows carry lengths (a.lengths) and each chain starts
// at its first real step. kSeqSeg: block (segment s, chain) walks steps
// [s seg_len, (s + 1) seg_len) from the state that the maps (A, U) of
// segments 0 .. s-1 (seg_reduce_kernel) carry h0 to. kSeqPlain keeps the
// plain scan's code.
// LATE: refill a consumed stage after the next stage's arithmetic (deep rings).
template <typename T, class M, int VEC, int R, int RB, bool GATED, int MODE, bool LATE>
__global__ void __launch_bounds__(32) seq_fwd_kernel(const __grid_constant__ SeqFwdArgs a) {
  constexpr bool VARLEN = MODE == kSeqVarlen, SEG = MODE == kSeqSeg;
  using IO = Io<T, VEC>;
  using G = typename GatePolicy<M>::type;
  constexpr int CHW = 32 * VEC;
  constexpr int NB = GATED ? 4 : 3;  // boxes per stage: x, rho, iota (, z)
  constexpr uint32_t BOX = seq_box_bytes<T, VEC, R>();
  static_assert(R % RB == 0, "kept states must fall on stage rows");
  // bfloat16 lanes without the merge run their arithmetic on packed pairs
  constexpr bool kPacked = G::kHalfInputs && VEC == 2 && !GATED;
  const Plan& p = a.p;
  extern __shared__ unsigned char seq_smem[];
  SeqRing<NB, BOX> ring{align128(seq_smem), nullptr, a.stages};
  ring.bars = reinterpret_cast<uint64_t*>(ring.stage(ring.S));

  const int lane = threadIdx.x;
  const int64_t n_g = (p.D + CHW - 1) / CHW;
  const int64_t chain = SEG ? blockIdx.x % p.n_chain : blockIdx.x;
  const int64_t sg = SEG ? blockIdx.x / p.n_chain : 0;
  const int64_t b = chain / n_g;
  const int64_t g = chain - b * n_g;
  const int64_t d0 = g * CHW + lane * VEC;
  const bool ch_ok = d0 < p.D;  // D % 8 == 0: a lane's VEC channels are all in or all out
  const int64_t BD = p.B * p.D;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);

  if (!SEG && blockIdx.x == 0)  // the segmented reduce kernel has done this
    seq_reset_workspace(a.ws, p, p.tag, lane);

  float k[VEC], kh[VEC], hc[VEC];
  const bool poly = seq_rates<VEC>(a.lambda, p.c, d0, ch_ok, k, kh);
#pragma unroll
  for (int v = 0; v < VEC; ++v) hc[v] = (ch_ok && a.h0 != nullptr) ? a.h0[b * p.D + d0 + v] : 0.0f;

  // The chain's steps: [t0, t0 + len) (all of them unless the rows carry
  // lengths or the chain is cut into segments).
  const int64_t t0 = SEG ? sg * p.seg_len : VARLEN ? row_start(a.lengths, b, p.L) : 0;
  const int64_t len = SEG ? min(p.seg_len, p.L - t0) : p.L - t0;
  const int64_t nblk = (len + R - 1) / R;
  const int cd = (int)(g * CHW), cb = (int)b;
  auto issue = [&](int st, int64_t j) {
    unsigned char* dst = ring.stage(st);
    const int t = (int)(t0 + j * R);
    mbar_arrive_expect_tx(&ring.bars[st], NB * BOX);
    tma_load_3d(dst, &a.tm_x, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + BOX, &a.tm_r, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + 2 * BOX, &a.tm_i, &ring.bars[st], cd, t, cb);
    if constexpr (GATED) tma_load_3d(dst + 3 * BOX, &a.tm_z, &ring.bars[st], cd, t, cb);
  };
  if (lane == 0) {
    for (int s = 0; s < ring.S; ++s) mbar_init(&ring.bars[s], 1);
    fence_mbar_init();
    for (int s = 0; s < ring.S && s < nblk; ++s) issue(s, s);
  }
  __syncwarp();
  if constexpr (SEG) {  // while the first stages load: the segment's start state
    if (ch_ok) seg_carry_in<VEC>(reinterpret_cast<const float2*>(a.ws + p.off_sagg) + b * p.D + d0,
                                 BD, sg, hc);
  }

  float* carry = reinterpret_cast<float*>(a.ws + (SEG ? p.off_skept : p.off_fpre)) + b * p.D + d0;
  int64_t cidx = SEG ? t0 / RB : 0;
  const int64_t n_carry = p.n_carry;
  int st = 0, prev = ring.S - 1;
  uint32_t phase = 0;
  for (int64_t j = 0; j < nblk; ++j) {
    mbar_wait(&ring.bars[st], phase, &fh->err);
    // Shallow rings refill the previous stage at the top of the iteration, deep
    // ones after this stage's arithmetic (as the backward).
    if (!LATE && lane == 0 && j > 0 && j - 1 + ring.S < nblk) {
      if (a.write_h) bulk_wait_read<0>();
      issue(prev, j - 1 + ring.S);
    }
    unsigned char* sb = ring.stage(st);
    unsigned char* lb = sb + lane * VEC * sizeof(T);
    const int64_t left = len - j * R;
    const int rows = (int)(left < R ? left : R);
    if constexpr (kPacked) {
      float2 hc2 = make_float2(hc[0], hc[1]);
      const float2 kh2 = make_float2(kh[0], kh[1]);
      if (rows == R) {
        if (poly)
          seq_fwd_stage_bf16x2<true, true, R, RB>(lb, rows, kh2, hc2, carry, cidx, n_carry, BD, ch_ok);
        else
          seq_fwd_stage_bf16x2<false, true, R, RB>(lb, rows, kh2, hc2, carry, cidx, n_carry, BD, ch_ok);
      } else {
        seq_fwd_stage_bf16x2<false, false, R, RB>(lb, rows, kh2, hc2, carry, cidx, n_carry, BD, ch_ok);
      }
      hc[0] = hc2.x;
      hc[1] = hc2.y;
    } else if (rows == R) {
      if (poly)
        seq_fwd_stage<IO, G, true, true, R, RB, GATED>(lb, rows, k, kh, hc, carry, cidx, n_carry, BD, ch_ok);
      else
        seq_fwd_stage<IO, G, false, true, R, RB, GATED>(lb, rows, k, kh, hc, carry, cidx, n_carry, BD, ch_ok);
    } else {
      seq_fwd_stage<IO, G, false, false, R, RB, GATED>(lb, rows, k, kh, hc, carry, cidx, n_carry, BD, ch_ok);
    }
    fence_proxy_async_smem();  // the stage's h rows, visible to the TMA store
    __syncwarp();
    if (lane == 0) {
      if (LATE && j > 0 && j - 1 + ring.S < nblk) {
        if (a.write_h) bulk_wait_read<0>();
        issue(prev, j - 1 + ring.S);
      }
      if (a.write_h) {
        tma_store_3d(&a.tm_h, sb, cd, (int)(t0 + j * R), cb);
        bulk_commit();
      }
    }
    prev = st;
    if (++st == ring.S) {
      st = 0;
      phase ^= 1u;
    }
  }
  if (lane == 0 && a.write_h) bulk_wait_all();
  if (a.h_last != nullptr && ch_ok && (!SEG || sg == p.nseg - 1)) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) a.h_last[b * p.D + d0 + v] = hc[v];
  }
}

// ----------------------------------------------------------------- backward

// One sub-block of RB steps (rows [0, srows) when not FULL) starting at row
// `row0` of the stage: forward recompute from the state hc, then the reverse
// recurrence carrying w = alpha g. dx, d rho and d iota overwrite dh, rho and
// iota of the same rows in the stage. GATED: the first box holds dy, the
// gradient of y = h SiLU(z) (Alg. 1), so dh = dy SiLU(z), and
// dz = dy h SiLU'(z) overwrites z in the fifth box.
template <class IO, class G, bool POLY, bool FULL, int R, int RB, bool GATED>
__device__ __forceinline__ void seq_bwd_sub(unsigned char* lb, int row0, int srows,
                                            const float (&k)[IO::VEC], const float (&kh)[IO::VEC],
                                            float (&hc)[IO::VEC], float (&w)[IO::VEC],
                                            float (&dlr)[IO::VEC]) {
  using Raw = typename IO::Raw;
  constexpr int V = IO::VEC;
  constexpr uint32_t ROWB = 32 * V * sizeof(typename IO::T);
  constexpr uint32_t BOX = R * ROWB;
  // boxes of a backward stage: dh (dy), x, rho, iota (, z)
  unsigned char* s_dh = lb + row0 * ROWB;
  const unsigned char* s_x = s_dh + BOX;
  unsigned char* s_r = s_dh + 2 * BOX;
  unsigned char* s_i = s_dh + 3 * BOX;
  unsigned char* s_z = s_dh + 4 * BOX;
  float E[RB][V], RS[RB][V], HP[RB][V];
#pragma unroll
  for (int s = 0; s < RB; ++s) {
    if (FULL || s < srows) {
      float xv[V], rv[V], iv[V], ix[V], l[V];
      if constexpr (G::kHalfInputs) {
        IO::unpack_half(*reinterpret_cast<const Raw*>(s_x + s * ROWB), xv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(s_r + s * ROWB), rv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(s_i + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          l[v] = G::decay_log_half(rv[v], kh[v]);
          ix[v] = G::gated_x_half(iv[v], xv[v]);
        }
      } else {
        IO::unpack(*reinterpret_cast<const Raw*>(s_x + s * ROWB), xv);
        IO::unpack(*reinterpret_cast<const Raw*>(s_r + s * ROWB), rv);
        IO::unpack(*reinterpret_cast<const Raw*>(s_i + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          l[v] = G::decay_log(rv[v], k[v], kh[v]);
          ix[v] = G::sigmoid(iv[v]) * xv[v];
        }
      }
#pragma unroll
      for (int v = 0; v < V; ++v) {
        const float e = expm1_neg<G::kDeg, POLY>(l[v]);
        const float q = -e * (e + 2.0f);
        const float rs = rsqrt_approx(fmaxf(q, 1e-30f));  // 1/sqrt(q); finite at q = 0
        E[s][v] = e;
        RS[s][v] = rs;
        HP[s][v] = hc[v];
        hc[v] = fmaf(1.0f + e, hc[v], (q * rs) * ix[v]);
      }
    }
  }
#pragma unroll
  for (int s = RB - 1; s >= 0; --s) {
    if (FULL || s < srows) {
      float gv[V], xv[V], rv[V], iv[V], ox[V], orho[V], oiota[V], sf[V], sdf[V], oz[V];
      IO::unpack(*reinterpret_cast<const Raw*>(s_dh + s * ROWB), gv);
      if constexpr (GATED) {
        float zv[V];
        if constexpr (G::kHalfInputs)
          IO::unpack_half(*reinterpret_cast<const Raw*>(s_z + s * ROWB), zv);
        else
          IO::unpack(*reinterpret_cast<const Raw*>(s_z + s * ROWB), zv);
#pragma unroll
        for (int v = 0; v < V; ++v) G::silu_grad(zv[v], sf[v], sdf[v]);
      }
      if constexpr (G::kHalfInputs) {  // bfloat16 pairs: re-read, not held from the recompute
        IO::unpack(lds_again(s_x + s * ROWB), xv);
        IO::unpack_half(lds_again(s_r + s * ROWB), rv);
        IO::unpack_half(lds_again(s_i + s * ROWB), iv);
      } else {
        IO::unpack(*reinterpret_cast<const Raw*>(s_x + s * ROWB), xv);
        IO::unpack(*reinterpret_cast<const Raw*>(s_r + s * ROWB), rv);
        IO::unpack(*reinterpret_cast<const Raw*>(s_i + s * ROWB), iv);
      }
#pragma unroll
      for (int v = 0; v < V; ++v) {
        const float e = E[s][v], rs = RS[s][v];
        const float alpha = 1.0f + e;
        const float q = -e * (e + 2.0f);
        float r, i;
        if constexpr (G::kHalfInputs) {
          r = G::sigmoid_half(rv[v]);
          i = G::sigmoid_half(iv[v]);
        } else {
          r = G::sigmoid(rv[v]);
          i = G::sigmoid(iv[v]);
        }
        float dhv = gv[v];
        if constexpr (GATED) dhv *= sf[v];
        const float g = dhv + w[v];
        w[v] = alpha * g;
        const float ix = i * xv[v];
        const float u = (q * rs) * ix;
        if constexpr (GATED) oz[v] = (gv[v] * fmaf(alpha, HP[s][v], u)) * sdf[v];  // dy h_t SiLU'
        ox[v] = (g * (q * rs)) * i;
        oiota[v] = (g * u) * (1.0f - i);
        // d/dl of h_t: alpha g (h_{t-1} - alpha u / q), with alpha g = w and
        // u / q = i x rs
        const float dl = w[v] * (HP[s][v] - (alpha * rs) * ix);
        orho[v] = (dl * k[v]) * fmaf(-r, r, r);
        dlr[v] = fmaf(dl, r, dlr[v]);
      }
      IO::store_smem(s_dh + s * ROWB, ox);
      IO::store_smem(s_r + s * ROWB, orho);
      IO::store_smem(s_i + s * ROWB, oiota);
      if constexpr (GATED) IO::store_smem(s_z + s * ROWB, oz);
    }
  }
}

// seq_bwd_sub for a bfloat16 lane under GatesFast, without the merge, on
// packed pairs. The forward recompute keeps, per step, alpha, -sqrt(1 - alpha^2)
// and c = h_{t-1} - alpha i x / sqrt(1 - alpha^2) (so that d l = alpha g c);
// the reverse recurrence re-reads the step's inputs for i and r, and uses
// r (1 - r) = (1 - tanh(rho/2)^2) / 4, so d rho = d l (k/4) (1 - tanh^2).
// kq = k/4 and nkq = -k/4 per channel.
template <bool POLY, bool FULL, int R, int RB>
__device__ __forceinline__ void seq_bwd_sub_bf16x2(unsigned char* lb, int row0, int srows, float2 kh,
                                                   float2 kq, float2 nkq, float2& hc, float2& w,
                                                   float2& dlr) {
  constexpr uint32_t ROWB = 128;
  constexpr uint32_t BOX = R * ROWB;
  unsigned char* s_dh = lb + row0 * ROWB;
  const unsigned char* s_x = s_dh + BOX;
  unsigned char* s_r = s_dh + 2 * BOX;
  unsigned char* s_i = s_dh + 3 * BOX;
  float2 AL[RB], NQ[RB], CP[RB];
#pragma unroll
  for (int s = 0; s < RB; ++s) {
    if (FULL || s < srows) {
      const float2 nhx = bf2_scaled(*reinterpret_cast<const uint32_t*>(s_x + s * ROWB), kBf2NegHalf);
      const float2 hr = bf2_scaled(*reinterpret_cast<const uint32_t*>(s_r + s * ROWB), kBf2Half);
      const float2 hi = bf2_scaled(*reinterpret_cast<const uint32_t*>(s_i + s * ROWB), kBf2Half);
      const float2 e = expm1_neg2<POLY>(__ffma2_rn(kh, tanh2(hr), kh));
      const float2 m2 = __fmul2_rn(e, __fadd2_rn(e, f2(2.0f)));  // -(1 - alpha^2)
      const float2 rs = make_float2(rsqrt_approx(fmaxf(-m2.x, 1e-30f)), rsqrt_approx(fmaxf(-m2.y, 1e-30f)));
      const float2 al = __fadd2_rn(f2(1.0f), e);
      const float2 nq = __fmul2_rn(m2, rs);                // -sqrt(1 - alpha^2)
      const float2 nix = __ffma2_rn(nhx, tanh2(hi), nhx);  // -i x
      AL[s] = al;
      NQ[s] = nq;
      CP[s] = __ffma2_rn(__fmul2_rn(al, rs), nix, hc);
      hc = __ffma2_rn(al, hc, __fmul2_rn(nq, nix));  // alpha h + sqrt(1 - alpha^2) i x
    }
  }
#pragma unroll
  for (int s = RB - 1; s >= 0; --s) {
    if (FULL || s < srows) {
      const float2 dh = bf2_unpack(*reinterpret_cast<const uint32_t*>(s_dh + s * ROWB));
      const float2 nhx = bf2_scaled(lds_again(s_x + s * ROWB), kBf2NegHalf);
      const float2 thr = tanh2(bf2_scaled(lds_again(s_r + s * ROWB), kBf2Half));
      const float2 thi = tanh2(bf2_scaled(lds_again(s_i + s * ROWB), kBf2Half));
      const float2 g = __fadd2_rn(dh, w);
      w = __fmul2_rn(AL[s], g);
      const float2 gnq = __fmul2_rn(g, NQ[s]);                    // -g sqrt(1 - alpha^2)
      const float2 ni = __ffma2_rn(f2(-0.5f), thi, f2(-0.5f));    // -i
      const float2 omi = __ffma2_rn(f2(-0.5f), thi, f2(0.5f));    // 1 - i
      const float2 nix = __ffma2_rn(nhx, thi, nhx);               // -i x
      const float2 ox = __fmul2_rn(gnq, ni);                      // g sqrt(1 - alpha^2) i
      const float2 oi = __fmul2_rn(__fmul2_rn(gnq, nix), omi);    // g u (1 - i)
      const float2 dl = __fmul2_rn(w, CP[s]);
      const float2 orho = __fmul2_rn(dl, __ffma2_rn(nkq, __fmul2_rn(thr, thr), kq));
      dlr = __ffma2_rn(dl, __ffma2_rn(f2(0.5f), thr, f2(0.5f)), dlr);  // += d l r
      *reinterpret_cast<uint32_t*>(s_dh + s * ROWB) = bf2_pack(ox);
      *reinterpret_cast<uint32_t*>(s_r + s * ROWB) = bf2_pack(orho);
      *reinterpret_cast<uint32_t*>(s_i + s * ROWB) = bf2_pack(oi);
    }
  }
}

// MODE as seq_fwd_kernel's. kSeqSeg: block (segment s, chain) starts from the
// adjoint carry that the maps (A, W) of the segments after s carry dh_last to,
// and only segment 0 writes dh0.
template <typename T, class M, int VEC, int R, int RB, bool GATED, int MODE, bool LATE>
__global__ void __launch_bounds__(32, sizeof(T) == 4 ? 8 : 16) seq_bwd_kernel(const __grid_constant__ SeqBwdArgs a) {
  constexpr bool VARLEN = MODE == kSeqVarlen, SEG = MODE == kSeqSeg;
  using IO = Io<T, VEC>;
  using G = typename GatePolicy<M>::type;
  constexpr int CHW = 32 * VEC;
  constexpr int NB = GATED ? 5 : 4;  // boxes per stage: dh (dy), x, rho, iota (, z)
  constexpr uint32_t BOX = seq_box_bytes<T, VEC, R>();
  constexpr int NSUB = R / RB;
  static_assert(R % RB == 0, "sub-blocks must tile a stage");
  constexpr bool kPacked = G::kHalfInputs && VEC == 2 && !GATED;  // as seq_fwd_kernel
  const Plan& p = a.p;
  extern __shared__ unsigned char seq_smem[];
  SeqRing<NB, BOX> ring{align128(seq_smem), nullptr, a.stages};
  ring.bars = reinterpret_cast<uint64_t*>(ring.stage(ring.S));

  const int lane = threadIdx.x;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(a.ws + p.off_bhdr);
  {
    int ok = 0;
    if (lane == 0) {
      ok = __ldcg(&fh->tag) == (SEG ? seg_tag(p.tag) : p.tag) && __ldcg(&fh->complete) == 1u;
      if (!ok) atomicOr(&fh->err, kErrWorkspace);
    }
    if (!__shfl_sync(kFull, ok, 0)) return;  // no forward states for this problem: write nothing
  }
  const int64_t n_g = (p.D + CHW - 1) / CHW;
  const int64_t chain = SEG ? blockIdx.x % p.n_chain : blockIdx.x;
  const int64_t sg = SEG ? blockIdx.x / p.n_chain : 0;
  const int64_t b = chain / n_g;
  const int64_t g = chain - b * n_g;
  const int64_t d0 = g * CHW + lane * VEC;
  const bool ch_ok = d0 < p.D;
  const int64_t BD = p.B * p.D;

  // The start states of the next QD sub-blocks, loaded QD sub-blocks ahead of
  // use (one ahead for bfloat16, whose registers are fully used).
  constexpr int QD = sizeof(T) == 4 ? 4 : 1;
  float k[VEC], kh[VEC], w[VEC], dlr[VEC], sq[QD][VEC];
  const bool poly = seq_rates<VEC>(a.lambda, p.c, d0, ch_ok, k, kh);
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    w[v] = (ch_ok && a.dh_last != nullptr) ? a.dh_last[b * p.D + d0 + v] : 0.0f;
    dlr[v] = 0.0f;
  }
  const int64_t t0 = SEG ? sg * p.seg_len : VARLEN ? row_start(a.lengths, b, p.L) : 0;
  const int64_t len = SEG ? min(p.seg_len, p.L - t0) : p.L - t0;
  const int64_t nblk = (len + R - 1) / R;
  const float* carry = reinterpret_cast<const float*>(a.ws + (SEG ? p.off_skept : p.off_fpre)) +
                       b * p.D + d0;
  const int64_t m0 = SEG ? t0 / RB : 0;  // kept states count from the chain's start
  // the state before sub-block m of this block: h0 for the chain's first, else
  // kept state m0 + m - 1
  auto load_start = [&](int64_t m, float (&out)[VEC]) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      out[v] = 0.0f;
      if (ch_ok) {
        if (m0 + m > 0)
          out[v] = __ldcg(carry + (m0 + m - 1) * BD + v);
        else if (a.h0 != nullptr)
          out[v] = a.h0[b * p.D + d0 + v];
      }
    }
  };
  const int cd = (int)(g * CHW), cb = (int)b;
  auto issue = [&](int st, int64_t j) {
    unsigned char* dst = ring.stage(st);
    const int t = (int)(t0 + j * R);
    mbar_arrive_expect_tx(&ring.bars[st], NB * BOX);
    tma_load_3d(dst, &a.tm_dh, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + BOX, &a.tm_x, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + 2 * BOX, &a.tm_r, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + 3 * BOX, &a.tm_i, &ring.bars[st], cd, t, cb);
    if constexpr (GATED) tma_load_3d(dst + 4 * BOX, &a.tm_z, &ring.bars[st], cd, t, cb);
  };
  if (lane == 0) {
    for (int s = 0; s < ring.S; ++s) mbar_init(&ring.bars[s], 1);
    fence_mbar_init();
    for (int s = 0; s < ring.S && s < nblk; ++s) issue(s, nblk - 1 - s);
  }
  __syncwarp();
  if constexpr (SEG) {  // while the first stages load: the segment's end carry
    if (ch_ok)
      seg_adjoint_in<VEC>(reinterpret_cast<const float2*>(a.ws + p.off_sagg) + b * p.D + d0, BD,
                          sg, p.nseg, w);
  }

  int64_t m = (len + RB - 1) / RB - 1;  // the sub-block processed next (-1: none)
#pragma unroll
  for (int u = 0; u < QD; ++u) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) sq[u][v] = 0.0f;
    if (m - u >= 0) load_start(m - u, sq[u]);
  }
  int st = 0, prev = ring.S - 1;
  uint32_t phase = 0;
  for (int64_t i = 0; i < nblk; ++i) {
    const int64_t j = nblk - 1 - i;
    mbar_wait(&ring.bars[st], phase, &fh->err);
    // Shallow rings refill the previous stage as soon as its stores have read
    // it, at the top of the iteration; deep ones after this stage's arithmetic,
    // when those stores are long done and the wait costs nothing.
    if (!LATE && lane == 0 && i > 0 && i - 1 + ring.S < nblk) {
      bulk_wait_read<0>();
      issue(prev, nblk - 1 - (i - 1 + ring.S));
    }
    unsigned char* sb = ring.stage(st);
    unsigned char* lb = sb + lane * VEC * sizeof(T);
    const int64_t left = len - j * R;
    const int rows = (int)(left < R ? left : R);
#pragma unroll
    for (int q = NSUB - 1; q >= 0; --q) {
      const int row0 = q * RB;
      if (row0 < rows) {
        const int srows = rows - row0 < RB ? rows - row0 : RB;
        float hc[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) hc[v] = sq[0][v];
#pragma unroll
        for (int u = 0; u + 1 < QD; ++u) {
#pragma unroll
          for (int v = 0; v < VEC; ++v) sq[u][v] = sq[u + 1][v];
        }
        if (m - QD >= 0) load_start(m - QD, sq[QD - 1]);  // in flight for QD sub-blocks
        if constexpr (kPacked) {
          float2 hc2 = make_float2(hc[0], hc[1]), w2 = make_float2(w[0], w[1]);
          float2 dlr2 = make_float2(dlr[0], dlr[1]);
          const float2 kh2 = make_float2(kh[0], kh[1]);
          const float2 kq = make_float2(0.25f * k[0], 0.25f * k[1]);
          const float2 nkq = make_float2(-kq.x, -kq.y);
          if (srows == RB) {
            if (poly)
              seq_bwd_sub_bf16x2<true, true, R, RB>(lb, row0, srows, kh2, kq, nkq, hc2, w2, dlr2);
            else
              seq_bwd_sub_bf16x2<false, true, R, RB>(lb, row0, srows, kh2, kq, nkq, hc2, w2, dlr2);
          } else {
            seq_bwd_sub_bf16x2<false, false, R, RB>(lb, row0, srows, kh2, kq, nkq, hc2, w2, dlr2);
          }
          w[0] = w2.x;
          w[1] = w2.y;
          dlr[0] = dlr2.x;
          dlr[1] = dlr2.y;
        } else if (srows == RB) {
          if (poly)
            seq_bwd_sub<IO, G, true, true, R, RB, GATED>(lb, row0, srows, k, kh, hc, w, dlr);
          else
            seq_bwd_sub<IO, G, false, true, R, RB, GATED>(lb, row0, srows, k, kh, hc, w, dlr);
        } else {
          seq_bwd_sub<IO, G, false, false, R, RB, GATED>(lb, row0, srows, k, kh, hc, w, dlr);
        }
        --m;
      }
    }
    fence_proxy_async_smem();  // the stage's outputs, visible to the TMA stores
    __syncwarp();
    if (lane == 0) {
      if (LATE && i > 0 && i - 1 + ring.S < nblk) {
        bulk_wait_read<0>();
        issue(prev, nblk - 1 - (i - 1 + ring.S));
      }
      const int t = (int)(t0 + j * R);
      tma_store_3d(&a.tm_dx, sb, cd, t, cb);
      tma_store_3d(&a.tm_dr, sb + 2 * BOX, cd, t, cb);
      tma_store_3d(&a.tm_di, sb + 3 * BOX, cd, t, cb);
      if constexpr (GATED) tma_store_3d(&a.tm_dz, sb + 4 * BOX, cd, t, cb);
      bulk_commit();
    }
    prev = st;
    if (++st == ring.S) {
      st = 0;
      phase ^= 1u;
    }
  }
  if (lane == 0) bulk_wait_all();

  double* acc = reinterpret_cast<double*>(a.ws + p.off_dlam);
  if (ch_ok) {
    if (a.dh0 != nullptr && (!SEG || sg == 0)) {
#pragma unroll
      for (int v = 0; v < VEC; ++v) a.dh0[b * p.D + d0 + v] = w[v];
    }
#pragma unroll
    for (int v = 0; v < VEC; ++v) atomicAdd(acc + (b % kStripes) * p.D + d0 + v, (double)dlr[v]);
  }
  // The last block out turns the partial sums into dLambda and clears them
  // (and the exit counter) for the next backward.
  __syncwarp();
  int last = 0;
  if (lane == 0) {
    __threadfence();
    last = atomicAdd(&bh->exited, 1u) == gridDim.x - 1;
  }
  if (__shfl_sync(kFull, last, 0)) {
    __threadfence();
    for (int64_t d = lane; d < p.D; d += 32) {
      double sum = 0.0;
      for (int s2 = 0; s2 < kStripes; ++s2) {
        sum += __ldcg(&acc[s2 * p.D + d]);
        acc[s2 * p.D + d] = 0.0;
      }
      const double lam = (double)a.lambda[d];
      const double sig = 1.0 / (1.0 + exp(-lam));  // d softplus / d Lambda
      a.dlambda[d] = (float)(-(double)p.c * sig * sum);
    }
    if (lane == 0) bh->exited = 0u;
  }
}

// ----------------------------------------------------- segment reductions

struct SegReduceArgs {
  CUtensorMap tm_a;  // forward: x; backward: dh (gated: dy)
  CUtensorMap tm_r;  // rho view
  CUtensorMap tm_i;  // forward: iota view
  CUtensorMap tm_z;  // gated backward: z
  Plan p;
  const float* lambda;
  unsigned char* ws;
  int stages;
};

// Rows [0, rows) of a forward reduce stage folded into the map (A, U): the
// gates as seq_fwd_stage evaluates them, then h -> alpha h + u composed after
// the map, step by step.
template <class IO, class G, bool POLY, bool FULL, int R>
__device__ __forceinline__ void seg_fold_fwd(const unsigned char* lb, int rows,
                                             const float (&k)[IO::VEC], const float (&kh)[IO::VEC],
                                             float (&A)[IO::VEC], float (&U)[IO::VEC]) {
  using Raw = typename IO::Raw;
  constexpr int V = IO::VEC;
  constexpr uint32_t ROWB = 32 * V * sizeof(typename IO::T);
  constexpr uint32_t BOX = R * ROWB;
#pragma unroll
  for (int s = 0; s < R; ++s) {
    if (FULL || s < rows) {
      float xv[V], rv[V], iv[V];
      if constexpr (G::kHalfInputs) {
        IO::unpack_half(*reinterpret_cast<const Raw*>(lb + s * ROWB), xv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(lb + BOX + s * ROWB), rv);
        IO::unpack_half(*reinterpret_cast<const Raw*>(lb + 2 * BOX + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          const float e = expm1_neg<G::kDeg, POLY>(G::decay_log_half(rv[v], kh[v]));
          const float u = G::sqrt(-e * (e + 2.0f)) * G::gated_x_half(iv[v], xv[v]);
          U[v] = fmaf(1.0f + e, U[v], u);
          A[v] *= 1.0f + e;
        }
      } else {
        IO::unpack(*reinterpret_cast<const Raw*>(lb + s * ROWB), xv);
        IO::unpack(*reinterpret_cast<const Raw*>(lb + BOX + s * ROWB), rv);
        IO::unpack(*reinterpret_cast<const Raw*>(lb + 2 * BOX + s * ROWB), iv);
#pragma unroll
        for (int v = 0; v < V; ++v) {
          const float e = expm1_neg<G::kDeg, POLY>(G::decay_log(rv[v], k[v], kh[v]));
          const float u = G::sqrt(-e * (e + 2.0f)) * (G::sigmoid(iv[v]) * xv[v]);
          U[v] = fmaf(1.0f + e, U[v], u);
          A[v] *= 1.0f + e;
        }
      }
    }
  }
}

// Rows [0, rows) of a backward reduce stage, last row first: w -> alpha (dh + w),
// and the product A of the alphas. GATED: the first box holds dy and the third
// z, and dh = dy SiLU(z).
template <class IO, class G, bool POLY, bool FULL, int R, bool GATED>
__device__ __forceinline__ void seg_fold_bwd(const unsigned char* lb, int rows,
                                             const float (&k)[IO::VEC], const float (&kh)[IO::VEC],
                                             float (&A)[IO::VEC], float (&w)[IO::VEC]) {
  using Raw = typename IO::Raw;
  constexpr int V = IO::VEC;
  constexpr uint32_t ROWB = 32 * V * sizeof(typename IO::T);
  constexpr uint32_t BOX = R * ROWB;
#pragma unroll
  for (int s = R - 1; s >= 0; --s) {
    if (FULL || s < rows) {
      float gv[V], rv[V], l[V];
      IO::unpack(*reinterpret_cast<const Raw*>(lb + s * ROWB), gv);
      if constexpr (GATED) {
        float zv[V];
        if constexpr (G::kHalfInputs)
          IO::unpack_half(*reinterpret_cast<const Raw*>(lb + 2 * BOX + s * ROWB), zv);
        else
          IO::unpack(*reinterpret_cast<const Raw*>(lb + 2 * BOX + s * ROWB), zv);
#pragma unroll
        for (int v = 0; v < V; ++v) gv[v] *= G::silu(zv[v]);
      }
      if constexpr (G::kHalfInputs) {
        IO::unpack_half(*reinterpret_cast<const Raw*>(lb + BOX + s * ROWB), rv);
#pragma unroll
        for (int v = 0; v < V; ++v) l[v] = G::decay_log_half(rv[v], kh[v]);
      } else {
        IO::unpack(*reinterpret_cast<const Raw*>(lb + BOX + s * ROWB), rv);
#pragma unroll
        for (int v = 0; v < V; ++v) l[v] = G::decay_log(rv[v], k[v], kh[v]);
      }
#pragma unroll
      for (int v = 0; v < V; ++v) {
        const float alpha = 1.0f + expm1_neg<G::kDeg, POLY>(l[v]);
        w[v] = alpha * (gv[v] + w[v]);
        A[v] *= alpha;
      }
    }
  }
}

// Segment reductions, one warp per (segment, chain) as the segmented serial
// kernels: the stage ring of those kernels without stores (a stage is
// refilled as soon as every lane has read it).
//   BWD = false: the forward map h_end = A h_start + U of the segment
//                (x, rho, iota in), stored at off_sagg; block 0 first restarts
//                the workspace bookkeeping for the forward.
//   BWD = true:  the adjoint map w_start = A w_end + W of the segment: A the
//                product of its alphas, W = w_start for w_end = 0 (dh, rho in;
//                GATED: dy, rho, z), stored at off_sagg over the forward's maps,
//                which only the forward call itself uses.
template <typename T, class M, int VEC, int R, bool BWD, bool GATED>
__global__ void __launch_bounds__(32) seg_reduce_kernel(const __grid_constant__ SegReduceArgs a) {
  static_assert(BWD || !GATED, "the forward map does not depend on z");
  using IO = Io<T, VEC>;
  using G = typename GatePolicy<M>::type;
  constexpr int CHW = 32 * VEC;
  constexpr int NB = (BWD && !GATED) ? 2 : 3;
  constexpr uint32_t BOX = seq_box_bytes<T, VEC, R>();
  const Plan& p = a.p;
  extern __shared__ unsigned char seq_smem[];
  SeqRing<NB, BOX> ring{align128(seq_smem), nullptr, a.stages};
  ring.bars = reinterpret_cast<uint64_t*>(ring.stage(ring.S));

  const int lane = threadIdx.x;
  const int64_t n_g = (p.D + CHW - 1) / CHW;
  const int64_t chain = blockIdx.x % p.n_chain;
  const int64_t sg = blockIdx.x / p.n_chain;
  const int64_t b = chain / n_g;
  const int64_t g = chain - b * n_g;
  const int64_t d0 = g * CHW + lane * VEC;
  const bool ch_ok = d0 < p.D;
  const int64_t BD = p.B * p.D;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  if (!BWD && blockIdx.x == 0) seq_reset_workspace(a.ws, p, seg_tag(p.tag), lane);

  float k[VEC], kh[VEC];
  const bool poly = seq_rates<VEC>(a.lambda, p.c, d0, ch_ok, k, kh);
  const int64_t t0 = sg * p.seg_len;
  const int64_t len = min(p.seg_len, p.L - t0);
  const int64_t nblk = (len + R - 1) / R;
  const int cd = (int)(g * CHW), cb = (int)b;
  // the forward takes the segment's stages in order, the backward from its end
  auto blk = [&](int64_t i) { return BWD ? nblk - 1 - i : i; };
  auto issue = [&](int st, int64_t j) {
    unsigned char* dst = ring.stage(st);
    const int t = (int)(t0 + j * R);
    mbar_arrive_expect_tx(&ring.bars[st], NB * BOX);
    tma_load_3d(dst, &a.tm_a, &ring.bars[st], cd, t, cb);
    tma_load_3d(dst + BOX, &a.tm_r, &ring.bars[st], cd, t, cb);
    if constexpr (!BWD) tma_load_3d(dst + 2 * BOX, &a.tm_i, &ring.bars[st], cd, t, cb);
    if constexpr (GATED) tma_load_3d(dst + 2 * BOX, &a.tm_z, &ring.bars[st], cd, t, cb);
  };
  if (lane == 0) {
    for (int s = 0; s < ring.S; ++s) mbar_init(&ring.bars[s], 1);
    fence_mbar_init();
    for (int s = 0; s < ring.S && s < nblk; ++s) issue(s, blk(s));
  }
  __syncwarp();

  float A[VEC], U[VEC];  // BWD: U is W
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    A[v] = 1.0f;
    U[v] = 0.0f;
  }
  int st = 0;
  uint32_t phase = 0;
  for (int64_t i = 0; i < nblk; ++i) {
    const int64_t j = blk(i);
    mbar_wait(&ring.bars[st], phase, &fh->err);
    const unsigned char* lb = ring.stage(st) + lane * VEC * sizeof(T);
    const int64_t left = len - j * R;
    const int rows = (int)(left < R ? left : R);
    if constexpr (BWD) {
      if (rows == R) {
        if (poly)
          seg_fold_bwd<IO, G, true, true, R, GATED>(lb, rows, k, kh, A, U);
        else
          seg_fold_bwd<IO, G, false, true, R, GATED>(lb, rows, k, kh, A, U);
      } else {
        seg_fold_bwd<IO, G, false, false, R, GATED>(lb, rows, k, kh, A, U);
      }
    } else {
      if (rows == R) {
        if (poly)
          seg_fold_fwd<IO, G, true, true, R>(lb, rows, k, kh, A, U);
        else
          seg_fold_fwd<IO, G, false, true, R>(lb, rows, k, kh, A, U);
      } else {
        seg_fold_fwd<IO, G, false, false, R>(lb, rows, k, kh, A, U);
      }
    }
    __syncwarp();  // every lane has read the stage: refill it
    if (lane == 0 && i + ring.S < nblk) issue(st, blk(i + ring.S));
    if (++st == ring.S) {
      st = 0;
      phase ^= 1u;
    }
  }
  if (ch_ok) {
    float2* out = reinterpret_cast<float2*>(a.ws + p.off_sagg) + sg * BD + b * p.D + d0;
#pragma unroll
    for (int v = 0; v < VEC; ++v) out[v] = make_float2(A[v], U[v]);
  }
}

}  // namespace blr
