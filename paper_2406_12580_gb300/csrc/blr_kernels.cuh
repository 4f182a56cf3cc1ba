// BD-LRU scan kernels for sm_103a: forward scan, backward reverse scan,
// single recurrent step. All are memory-bound elementwise scans: no tensor
// cores, 16-byte loads and stores along the channels, gate arithmetic fused
// into the load, float32 state.
//
// Scan structure (one thread block per tile of ttile steps x dblk channels):
//   1. each thread loads its tc x vec elements, computes the gates and folds
//      its chunk into one affine map h -> A h + U (serial, in registers);
//   2. warp 0 turns the chunk maps of every channel into exclusive prefix maps
//      (shared memory) and the tile's total map;
//   3. warp 0 chains the tile to its predecessors in time with a decoupled
//      look-back over per-tile records in the workspace (bounded waits);
//   4. every thread applies its prefix map to the tile's carry and re-runs its
//      chunk from the true state, writing the outputs.
// Tiles are handed out in launch order by an atomic ticket, time-major, so a
// block only ever waits for blocks that started before it.
#pragma once

#include "blr_device.cuh"

namespace blr {

struct FwdArgs {
  Plan p;
  const void* x;
  const void* gl;
  const float* lambda;
  const float* h0;
  void* h;
  float* h_last;
  unsigned char* ws;
};

struct BwdArgs {
  Plan p;
  const void* dh;
  const float* dh_last;
  const void* x;
  const void* gl;
  const float* lambda;
  const float* h0;
  void* dx;
  void* dgl;
  float* dlambda;
  float* dh0;
  unsigned char* ws;
};

struct StepArgs {
  int64_t B, D;
  float c;
  int rows;          // batch rows per thread
  int64_t n_vgroups; // blocks along the channel vectors
  const float* h_prev;
  const void* x;
  const void* gl;
  const float* lambda;
  float* h_t;
};

constexpr int kCpl = kMaxDblk / 32;  // channels per lane of warp 0

// ---------------------------------------------------------------- forward scan

template <class IO, class M>
__global__ void __launch_bounds__(256) scan_fwd_kernel(const FwdArgs a) {
  constexpr int VEC = IO::kVec;
  constexpr int TC = kTc;
  using T = typename IO::T;
  const Plan& p = a.p;

  __shared__ float2 s_map[kMaxNt][kMaxDblk];  // chunk map, then exclusive prefix map
  __shared__ float s_carry[kMaxDblk];
  __shared__ uint32_t s_ticket;

  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  uint32_t* flags = reinterpret_cast<uint32_t*>(a.ws + p.off_fflags);
  float2* agg = reinterpret_cast<float2*>(a.ws + p.off_fagg);
  float* pre = reinterpret_cast<float*>(a.ws + p.off_fpre);

  const int tx = threadIdx.x, ty = threadIdx.y;
  const int tid = ty * p.nv + tx;
  if (tid == 0) s_ticket = atomicAdd(&fh->ticket, 1u);
  __syncthreads();
  const int64_t rec = s_ticket;
  const int64_t it = rec / p.n_c;
  const int64_t cb = rec - it * p.n_c;
  const int64_t b = cb / p.n_dblk;
  const int64_t dbase = (cb - b * p.n_dblk) * p.dblk;
  const int cl = tx * VEC;
  const int64_t d0 = dbase + cl;
  const bool ch_ok = d0 < p.D;
  const int64_t t0 = it * p.ttile + (int64_t)ty * TC;
  if (rec == 0 && tid == 0) fh->tag = p.tag;

  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);

  float k[VEC];
#pragma unroll
  for (int j = 0; j < VEC; j += 4) {
    float lam[4] = {0.f, 0.f, 0.f, 0.f};
    if (ch_ok) load_f32x4(a.lambda + d0 + j, lam);
#pragma unroll
    for (int v = 0; v < 4; ++v) k[j + v] = decay_rate(p.c, lam[v]);
  }

  // 1. loads (all issued before any use), gates, chunk map.
  float xv[TC][VEC], rv[TC][VEC], iv[TC][VEC];
#pragma unroll
  for (int s = 0; s < TC; ++s) {
    const int64_t t = t0 + s;
    if (ch_ok && t < p.L) {
      const int64_t row = b * p.L + t;
      IO::load(x + row * p.D + d0, xv[s]);
      IO::load(gl + row * 2 * p.D + d0, rv[s]);
      IO::load(gl + row * 2 * p.D + p.D + d0, iv[s]);
    }
  }
  float al[TC][VEC], u[TC][VEC];
#pragma unroll
  for (int s = 0; s < TC; ++s) {
    const bool ok = ch_ok && (t0 + s < p.L);
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      if (ok) {
        float r, i, alpha, q;
        gates<M>(k[v], rv[s][v], iv[s][v], r, i, alpha, q);
        al[s][v] = alpha;
        u[s][v] = M::sqrt(q) * i * xv[s][v];
      } else {  // outside the sequence or the channels: the identity map
        al[s][v] = 1.0f;
        u[s][v] = 0.0f;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    float A = 1.0f, U = 0.0f;
#pragma unroll
    for (int s = 0; s < TC; ++s) {
      U = fmaf(al[s][v], U, u[s][v]);
      A *= al[s][v];
    }
    s_map[ty][cl + v] = make_float2(A, U);
  }
  __syncthreads();

  // 2.-3. warp 0: prefix maps, tile map, look-back, tile prefix.
  if (tid < 32) {
    uint32_t* err = &fh->err;
    float tA[kCpl], tU[kCpl], carry[kCpl];
#pragma unroll
    for (int j = 0; j < kCpl; ++j) {
      const int ch = tid + 32 * j;
      float pa = 1.0f, pu = 0.0f;
      if (ch < p.dblk) {
        for (int m = 0; m < p.nt; ++m) {
          const float2 e = s_map[m][ch];
          s_map[m][ch] = make_float2(pa, pu);
          pu = fmaf(e.x, pu, e.y);
          pa *= e.x;
        }
      }
      tA[j] = pa;
      tU[j] = pu;
      carry[j] = 0.0f;
    }
    if (it == 0) {
#pragma unroll
      for (int j = 0; j < kCpl; ++j) {
        const int ch = tid + 32 * j;
        if (ch < p.dblk && dbase + ch < p.D && a.h0 != nullptr) carry[j] = a.h0[b * p.D + dbase + ch];
      }
    } else {
#pragma unroll
      for (int j = 0; j < kCpl; ++j) {
        const int ch = tid + 32 * j;
        if (ch < p.dblk) __stcg(&agg[rec * p.dblk + ch], make_float2(tA[j], tU[j]));
      }
      __threadfence();
      __syncwarp();
      if (tid == 0) st_release(&flags[rec], kFlagAggregate);
      float ea[kCpl], eu[kCpl];
#pragma unroll
      for (int j = 0; j < kCpl; ++j) { ea[j] = 1.0f; eu[j] = 0.0f; }
      int64_t q = rec - p.n_c;  // the same channel block, one tile earlier
      for (;;) {
        const uint32_t f = wait_flag(&flags[q], err, kWaitTimeoutNs);
        if (f != kFlagAggregate) {  // a prefix (or 0: the wait expired, carry 0)
#pragma unroll
          for (int j = 0; j < kCpl; ++j) {
            const int ch = tid + 32 * j;
            if (ch < p.dblk) {
              const float pv = (f == kFlagPrefix) ? __ldcg(&pre[q * p.dblk + ch]) : 0.0f;
              carry[j] = fmaf(ea[j], pv, eu[j]);
            }
          }
          break;
        }
#pragma unroll
        for (int j = 0; j < kCpl; ++j) {
          const int ch = tid + 32 * j;
          if (ch < p.dblk) {
            const float2 g = __ldcg(&agg[q * p.dblk + ch]);
            eu[j] = fmaf(ea[j], g.y, eu[j]);
            ea[j] *= g.x;
          }
        }
        q -= p.n_c;
      }
    }
#pragma unroll
    for (int j = 0; j < kCpl; ++j) {
      const int ch = tid + 32 * j;
      if (ch < p.dblk) {
        const float incl = fmaf(tA[j], carry[j], tU[j]);
        __stcg(&pre[rec * p.dblk + ch], incl);
        s_carry[ch] = carry[j];
        if (it == p.n_t - 1 && a.h_last != nullptr && dbase + ch < p.D)
          a.h_last[b * p.D + dbase + ch] = incl;
      }
    }
    __threadfence();
    __syncwarp();
    if (tid == 0) st_release(&flags[rec], kFlagPrefix);
  }
  __syncthreads();

  // 4. re-run the chunk from its true starting state.
  if (a.h != nullptr && ch_ok) {
    T* h = static_cast<T*>(a.h);
    float hs[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const float2 m = s_map[ty][cl + v];
      hs[v] = fmaf(m.x, s_carry[cl + v], m.y);
    }
#pragma unroll
    for (int s = 0; s < TC; ++s) {
      float out[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        hs[v] = fmaf(al[s][v], hs[v], u[s][v]);
        out[v] = hs[v];
      }
      const int64_t t = t0 + s;
      if (t < p.L) IO::store(h + (b * p.L + t) * p.D + d0, out);
    }
  }
  if (tid == 0) atomicAdd(&fh->done, 1u);
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

template <class IO, class M>
__global__ void __launch_bounds__(256) scan_bwd_kernel(const BwdArgs a) {
  constexpr int VEC = IO::kVec;
  constexpr int TC = kTc;
  using T = typename IO::T;
  const Plan& p = a.p;

  __shared__ float s_a[kMaxNt][kMaxDblk];   // chunk prod alpha -> prefix map A
  __shared__ float s_u[kMaxNt][kMaxDblk];   // chunk U          -> prefix map U
  __shared__ float s_w[kMaxNt][kMaxDblk];   // chunk W          -> suffix map W
  __shared__ float s_sa[kMaxNt][kMaxDblk];  //                  -> suffix map A
  __shared__ float s_hc[kMaxDblk], s_wc[kMaxDblk];
  __shared__ uint32_t s_ticket;
  __shared__ int s_flag;

  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(a.ws + p.off_bhdr);
  uint32_t* flags = reinterpret_cast<uint32_t*>(a.ws + p.off_bflags);
  float2* agg = reinterpret_cast<float2*>(a.ws + p.off_bagg);
  float* pre = reinterpret_cast<float*>(a.ws + p.off_bpre);
  const float* fpre = reinterpret_cast<const float*>(a.ws + p.off_fpre);
  double* dlam_acc = reinterpret_cast<double*>(a.ws + p.off_dlam);

  const int tx = threadIdx.x, ty = threadIdx.y;
  const int tid = ty * p.nv + tx;
  const int nthreads = p.nv * p.nt;
  if (tid == 0) {
    s_ticket = atomicAdd(&bh->ticket, 1u);
    const bool ok = __ldcg(&fh->tag) == p.tag && __ldcg(&fh->done) == (uint32_t)p.n_tiles;
    if (!ok) atomicOr(&fh->err, kErrWorkspace);
    s_flag = ok;
  }
  __syncthreads();
  if (!s_flag) return;  // no forward carries for this problem: write nothing
  const int64_t ticket = s_ticket;
  const int64_t it = p.n_t - 1 - ticket / p.n_c;  // tiles handed out from the end
  const int64_t cb = ticket % p.n_c;
  const int64_t rec = it * p.n_c + cb;
  const int64_t b = cb / p.n_dblk;
  const int64_t dbase = (cb - b * p.n_dblk) * p.dblk;
  const int cl = tx * VEC;
  const int64_t d0 = dbase + cl;
  const bool ch_ok = d0 < p.D;
  const int64_t t0 = it * p.ttile + (int64_t)ty * TC;

  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);
  const T* dh = static_cast<const T*>(a.dh);

  float k[VEC];
#pragma unroll
  for (int j = 0; j < VEC; j += 4) {
    float lam[4] = {0.f, 0.f, 0.f, 0.f};
    if (ch_ok) load_f32x4(a.lambda + d0 + j, lam);
#pragma unroll
    for (int v = 0; v < 4; ++v) k[j + v] = decay_rate(p.c, lam[v]);
  }

  // 1. loads, gates, chunk maps of both directions.
  float xv[TC][VEC], rv[TC][VEC], iv[TC][VEC], gv[TC][VEC];
#pragma unroll
  for (int s = 0; s < TC; ++s) {
    const int64_t t = t0 + s;
    if (ch_ok && t < p.L) {
      const int64_t row = b * p.L + t;
      IO::load(dh + row * p.D + d0, gv[s]);
      IO::load(x + row * p.D + d0, xv[s]);
      IO::load(gl + row * 2 * p.D + d0, rv[s]);
      IO::load(gl + row * 2 * p.D + p.D + d0, iv[s]);
    }
  }
  // Per element kept for the last pass: alpha, u, beta = n i, c2 = alpha u / q,
  // ui = u (1 - i), r, and dh (then g).
  float al[TC][VEC], u[TC][VEC], bt[TC][VEC], c2[TC][VEC], ui[TC][VEC], rr[TC][VEC];
#pragma unroll
  for (int s = 0; s < TC; ++s) {
    const bool ok = ch_ok && (t0 + s < p.L);
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      if (ok) {
        float r, i, alpha, q;
        gates<M>(k[v], rv[s][v], iv[s][v], r, i, alpha, q);
        const float beta = M::sqrt(q) * i;
        const float uu = beta * xv[s][v];
        al[s][v] = alpha;
        u[s][v] = uu;
        bt[s][v] = beta;
        c2[s][v] = M::div(alpha * uu, q);
        ui[s][v] = uu * (1.0f - i);
        rr[s][v] = r;
      } else {
        al[s][v] = 1.0f;
        u[s][v] = 0.0f;
        bt[s][v] = 0.0f;
        c2[s][v] = 0.0f;
        ui[s][v] = 0.0f;
        rr[s][v] = 0.0f;
        gv[s][v] = 0.0f;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    float A = 1.0f, U = 0.0f, W = 0.0f;
#pragma unroll
    for (int s = 0; s < TC; ++s) {
      U = fmaf(al[s][v], U, u[s][v]);
      A *= al[s][v];            // prod of alpha up to and including s
      W = fmaf(A, gv[s][v], W); // w at the chunk start from a zero carry
    }
    s_a[ty][cl + v] = A;
    s_u[ty][cl + v] = U;
    s_w[ty][cl + v] = W;
  }
  __syncthreads();

  // 2.-3. warp 0.
  if (tid < 32) {
    uint32_t* err = &fh->err;
    float tA[kCpl], tW[kCpl], hc[kCpl], wc[kCpl];
#pragma unroll
    for (int j = 0; j < kCpl; ++j) {
      const int ch = tid + 32 * j;
      float sa = 1.0f, su = 0.0f;
      if (ch < p.dblk) {
        for (int m = p.nt - 1; m >= 0; --m) {  // suffix maps, from the tile's end
          const float A = s_a[m][ch], W = s_w[m][ch];
          s_sa[m][ch] = sa;
          s_w[m][ch] = su;
          su = fmaf(A, su, W);
          sa *= A;
        }
        float pa = 1.0f, pu = 0.0f;
        for (int m = 0; m < p.nt; ++m) {       // prefix maps, from the tile's start
          const float A = s_a[m][ch], U = s_u[m][ch];
          s_a[m][ch] = pa;
          s_u[m][ch] = pu;
          pu = fmaf(A, pu, U);
          pa *= A;
        }
      }
      tA[j] = sa;
      tW[j] = su;
      hc[j] = 0.0f;
      wc[j] = 0.0f;
      if (ch < p.dblk && dbase + ch < p.D) {
        if (it > 0)
          hc[j] = __ldcg(&fpre[(rec - p.n_c) * p.dblk + ch]);
        else if (a.h0 != nullptr)
          hc[j] = a.h0[b * p.D + dbase + ch];
      }
    }
    if (it == p.n_t - 1) {
#pragma unroll
      for (int j = 0; j < kCpl; ++j) {
        const int ch = tid + 32 * j;
        if (ch < p.dblk && dbase + ch < p.D && a.dh_last != nullptr)
          wc[j] = a.dh_last[b * p.D + dbase + ch];
      }
    } else {
#pragma unroll
      for (int j = 0; j < kCpl; ++j) {
        const int ch = tid + 32 * j;
        if (ch < p.dblk) __stcg(&agg[rec * p.dblk + ch], make_float2(tA[j], tW[j]));
      }
      __threadfence();
      __syncwarp();
      if (tid == 0) st_release(&flags[rec], kFlagAggregate);
      float ea[kCpl], eu[kCpl];
#pragma unroll
      for (int j = 0; j < kCpl; ++j) { ea[j] = 1.0f; eu[j] = 0.0f; }
      int64_t q = rec + p.n_c;  // the same channel block, one tile later
      for (;;) {
        const uint32_t f = wait_flag(&flags[q], err, kWaitTimeoutNs);
        if (f != kFlagAggregate) {
#pragma unroll
          for (int j = 0; j < kCpl; ++j) {
            const int ch = tid + 32 * j;
            if (ch < p.dblk) {
              const float pv = (f == kFlagPrefix) ? __ldcg(&pre[q * p.dblk + ch]) : 0.0f;
              wc[j] = fmaf(ea[j], pv, eu[j]);
            }
          }
          break;
        }
#pragma unroll
        for (int j = 0; j < kCpl; ++j) {
          const int ch = tid + 32 * j;
          if (ch < p.dblk) {
            const float2 g = __ldcg(&agg[q * p.dblk + ch]);
            eu[j] = fmaf(ea[j], g.y, eu[j]);
            ea[j] *= g.x;
          }
        }
        q += p.n_c;
      }
    }
#pragma unroll
    for (int j = 0; j < kCpl; ++j) {
      const int ch = tid + 32 * j;
      if (ch < p.dblk) {
        const float incl = fmaf(tA[j], wc[j], tW[j]);  // w at the tile's first step
        __stcg(&pre[rec * p.dblk + ch], incl);
        s_hc[ch] = hc[j];
        s_wc[ch] = wc[j];
        if (it == 0 && a.dh0 != nullptr && dbase + ch < p.D) a.dh0[b * p.D + dbase + ch] = incl;
      }
    }
    __threadfence();
    __syncwarp();
    if (tid == 0) st_release(&flags[rec], kFlagPrefix);
  }
  __syncthreads();

  // 4. g backwards through the chunk, then the gradients forwards with h_{t-1}.
  float hs[VEC], wn[VEC], dl_r[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    hs[v] = fmaf(s_a[ty][cl + v], s_hc[cl + v], s_u[ty][cl + v]);
    wn[v] = fmaf(s_sa[ty][cl + v], s_wc[cl + v], s_w[ty][cl + v]);
    dl_r[v] = 0.0f;
  }
#pragma unroll
  for (int s = TC - 1; s >= 0; --s) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const float g = gv[s][v] + wn[v];
      gv[s][v] = g;
      wn[v] = al[s][v] * g;
    }
  }
  T* dx = static_cast<T*>(a.dx);
  T* dgl = static_cast<T*>(a.dgl);
#pragma unroll
  for (int s = 0; s < TC; ++s) {
    float ox[VEC], orho[VEC], oiota[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const float g = gv[s][v];
      const float dl = g * al[s][v] * (hs[v] - c2[s][v]);
      const float r = rr[s][v];
      orho[v] = dl * k[v] * (r - r * r);
      oiota[v] = g * ui[s][v];
      ox[v] = g * bt[s][v];
      dl_r[v] = fmaf(dl, r, dl_r[v]);
      hs[v] = fmaf(al[s][v], hs[v], u[s][v]);
    }
    const int64_t t = t0 + s;
    if (ch_ok && t < p.L) {
      const int64_t row = b * p.L + t;
      IO::store(dx + row * p.D + d0, ox);
      IO::store(dgl + row * 2 * p.D + d0, orho);
      IO::store(dgl + row * 2 * p.D + p.D + d0, oiota);
    }
  }

  // 5. dLambda: block sum over time chunks, float64 stripes, last block finishes.
  __syncthreads();  // s_a is reused
#pragma unroll
  for (int v = 0; v < VEC; ++v) s_a[ty][cl + v] = dl_r[v];
  __syncthreads();
  if (ty == 0 && ch_ok) {
    const int stripe = (int)(b % kStripes);
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      float sum = 0.0f;
      for (int m = 0; m < p.nt; ++m) sum += s_a[m][cl + v];
      atomicAdd(&dlam_acc[stripe * p.D + d0 + v], (double)sum);
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(&bh->done, 1u) == (uint32_t)(p.n_tiles - 1));
  __syncthreads();
  if (s_flag) {
    __threadfence();
    for (int64_t d = tid; d < p.D; d += nthreads) {
      double sum = 0.0;
      for (int st = 0; st < kStripes; ++st) sum += __ldcg(&dlam_acc[st * p.D + d]);
      const double lam = (double)a.lambda[d];
      const double sig = 1.0 / (1.0 + exp(-lam));  // d softplus / d Lambda
      a.dlambda[d] = (float)(-(double)p.c * sig * sum);
    }
  }
}

// ------------------------------------------------------------ recurrent step

template <class IO, class M, int ROWS>
__global__ void __launch_bounds__(256) step_kernel(const StepArgs a) {
  constexpr int VEC = IO::kVec;
  using T = typename IO::T;
  const int64_t nvec = a.D / VEC;
  const int64_t vg = blockIdx.x % a.n_vgroups;
  const int64_t rg = blockIdx.x / a.n_vgroups;
  const int64_t vi = vg * blockDim.x + threadIdx.x;
  if (vi >= nvec) return;
  const int64_t d0 = vi * VEC;
  const int64_t r0 = (rg * blockDim.y + threadIdx.y) * ROWS;

  float k[VEC];
#pragma unroll
  for (int j = 0; j < VEC; j += 4) {
    float lam[4];
    load_f32x4(a.lambda + d0 + j, lam);
#pragma unroll
    for (int v = 0; v < 4; ++v) k[j + v] = decay_rate(a.c, lam[v]);
  }
  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);
  float hp[ROWS][VEC], xv[ROWS][VEC], rv[ROWS][VEC], iv[ROWS][VEC];
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const int64_t bb = r0 + r;
    if (bb < a.B) {
#pragma unroll
      for (int j = 0; j < VEC; j += 4) load_f32x4(a.h_prev + bb * a.D + d0 + j, &hp[r][j]);
      IO::load(x + bb * a.D + d0, xv[r]);
      IO::load(gl + bb * 2 * a.D + d0, rv[r]);
      IO::load(gl + bb * 2 * a.D + a.D + d0, iv[r]);
    }
  }
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    const int64_t bb = r0 + r;
    if (bb < a.B) {
      float out[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        float rg_, i, alpha, q;
        gates<M>(k[v], rv[r][v], iv[r][v], rg_, i, alpha, q);
        out[v] = fmaf(alpha, hp[r][v], M::sqrt(q) * i * xv[r][v]);
      }
#pragma unroll
      for (int j = 0; j < VEC; j += 4)
        *reinterpret_cast<float4*>(a.h_t + bb * a.D + d0 + j) =
            make_float4(out[j], out[j + 1], out[j + 2], out[j + 3]);
    }
  }
}

// ------------------------------------------------------------ bounded-wait test

__global__ void selftest_wait_kernel(const uint32_t* flag, uint32_t* err, uint64_t timeout_ns) {
  (void)wait_flag(flag, err, timeout_ns);
}

}  // namespace blr
