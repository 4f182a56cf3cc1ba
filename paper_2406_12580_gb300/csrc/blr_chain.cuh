// Warp-chain scan kernels: the BD-LRU scan when a problem has enough
// independent (batch row, channel group) chains to fill the GPU on its own.
//
// One warp owns CH = NVL * 4 channels of one batch row and walks the whole
// sequence in blocks of BS = NTL * kTc steps (lanes: NVL along channels x NTL
// along time, kTc steps each). Inside a block the lanes' chunk maps are
// combined with warp shuffles (the first-order linear scan of Sec. 3.3); the
// state between blocks stays in registers. There is no look-back, no barrier
// and no shared memory; the next block's inputs are loaded while the current
// one is computed. The forward writes the state after every block, which the
// backward uses as its h carries; the backward walks the blocks from the end,
// carrying w = alpha g.
#pragma once

#include "blr_kernels.cuh"

namespace blr {

struct ChainFwdArgs {
  Plan p;
  const void* x;
  const void* gl;
  const float* h0;
  void* h;
  float* h_last;
  unsigned char* ws;
};

struct ChainBwdArgs {
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

// Prefix / suffix combine over the NTL time lanes of a warp (lane = tcl * NVL + cv).
template <int NVL, int V>
__device__ __forceinline__ void chain_prefix(float (&A)[V], float (&U)[V], int tcl, float (&ea)[V],
                                             float (&eu)[V]) {
  constexpr int NTL = 32 / NVL;
#pragma unroll
  for (int off = 1; off < NTL; off <<= 1) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float pa = __shfl_up_sync(kFull, A[v], off * NVL);
      const float pu = __shfl_up_sync(kFull, U[v], off * NVL);
      if (tcl >= off) {
        U[v] = fmaf(A[v], pu, U[v]);
        A[v] *= pa;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    ea[v] = __shfl_up_sync(kFull, A[v], NVL);
    eu[v] = __shfl_up_sync(kFull, U[v], NVL);
    if (tcl == 0) {
      ea[v] = 1.0f;
      eu[v] = 0.0f;
    }
  }
}

template <int NVL, int V>
__device__ __forceinline__ void chain_suffix(float (&A)[V], float (&W)[V], int tcl, float (&sa)[V],
                                             float (&sw)[V]) {
  constexpr int NTL = 32 / NVL;
#pragma unroll
  for (int off = 1; off < NTL; off <<= 1) {
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float na = __shfl_down_sync(kFull, A[v], off * NVL);
      const float nw = __shfl_down_sync(kFull, W[v], off * NVL);
      if (tcl + off < NTL) {
        W[v] = fmaf(A[v], nw, W[v]);
        A[v] *= na;
      }
    }
  }
#pragma unroll
  for (int v = 0; v < V; ++v) {
    sa[v] = __shfl_down_sync(kFull, A[v], NVL);
    sw[v] = __shfl_down_sync(kFull, W[v], NVL);
    if (tcl == NTL - 1) {
      sa[v] = 1.0f;
      sw[v] = 0.0f;
    }
  }
}

// ------------------------------------------------------------------ forward

template <typename T, class M, int NVL>
__global__ void __launch_bounds__(128) chain_fwd_kernel(const ChainFwdArgs a) {
  using IO = Io<T, 4>;
  using Raw = typename IO::Raw;
  constexpr int VEC = 4;
  constexpr int NTL = 32 / NVL;
  constexpr int CH = NVL * VEC;
  constexpr int BS = NTL * kTc;
  const Plan& p = a.p;
  const int lane = threadIdx.x & 31;
  const int64_t wid = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t n_cg = (p.D + CH - 1) / CH;
  const bool warp_ok = wid < p.B * n_cg;  // surplus warps of the last block idle
  const int64_t b = warp_ok ? wid / n_cg : 0;
  const int64_t d0 = warp_ok ? (wid - b * n_cg) * CH + (lane % NVL) * VEC : p.D;
  const int tcl = lane / NVL;
  const bool ch_ok = d0 < p.D;
  const int64_t BD = p.B * p.D;
  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);
  T* h = static_cast<T*>(a.h);
  uint32_t* pre = reinterpret_cast<uint32_t*>(a.ws + p.off_fpre);
  const float* kd = reinterpret_cast<const float*>(a.ws + p.off_k);

  float k[VEC], carry[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    k[v] = 0.0f;
    carry[v] = 0.0f;
  }
  if (ch_ok) {
    load_f32<VEC>(kd + d0, k);
    if (a.h0 != nullptr) load_f32<VEC>(a.h0 + b * p.D + d0, carry);
  }
  const int64_t nblk = warp_ok ? (p.L + BS - 1) / BS : 0;
  Raw rx[kTc], rr[kTc], ri[kTc];
  auto fetch = [&](int64_t j) {
    const int64_t t0 = j * BS + tcl * kTc;
    if (!ch_ok) return;
    const T* px = x + (b * p.L + t0) * p.D + d0;
    const T* pg = gl + (b * p.L + t0) * 2 * p.D + d0;
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      if (t0 + s < p.L) {
        rx[s] = IO::load_raw(px + s * p.D);
        rr[s] = IO::load_raw(pg + s * 2 * p.D);
        ri[s] = IO::load_raw(pg + s * 2 * p.D + p.D);
      }
    }
  };
  if (nblk > 0) fetch(0);
  for (int64_t j = 0; j < nblk; ++j) {
    const int64_t t0 = j * BS + tcl * kTc;
    const int64_t left = ch_ok ? p.L - t0 : 0;
    const int valid = (int)(left < 0 ? 0 : (left > kTc ? kTc : left));
    float al[kTc][VEC], u[kTc][VEC];
    if (valid == kTc)
      fwd_chunk<IO, M, true>(k, rx, rr, ri, valid, al, u);
    else
      fwd_chunk<IO, M, false>(k, rx, rr, ri, valid, al, u);
    if (j + 1 < nblk) fetch(j + 1);  // the next block's loads overlap this block
    float A[VEC], U[VEC], ea[VEC], eu[VEC];
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
    chain_prefix<NVL, VEC>(A, U, tcl, ea, eu);
    float hs[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) hs[v] = fmaf(ea[v], carry[v], eu[v]);
    T* ph = h + (b * p.L + t0) * p.D + d0;
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      float out[VEC];
#pragma unroll
      for (int v = 0; v < VEC; ++v) {
        hs[v] = fmaf(al[s][v], hs[v], u[s][v]);
        out[v] = hs[v];
      }
      if (h != nullptr && s < valid) IO::store(ph + s * p.D, out);
    }
    // the state after the block: the last time lane's inclusive map on the carry
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const float fa = __shfl_sync(kFull, A[v], (NTL - 1) * NVL + lane % NVL);
      const float fu = __shfl_sync(kFull, U[v], (NTL - 1) * NVL + lane % NVL);
      carry[v] = fmaf(fa, carry[v], fu);
    }
    if (tcl == NTL - 1 && ch_ok && j + 1 < nblk) {  // the backward's h carry of block j + 1
#pragma unroll
      for (int v = 0; v < VEC; ++v) pre[j * BD + b * p.D + d0 + v] = __float_as_uint(carry[v]);
    }
  }
  if (warp_ok && a.h_last != nullptr && tcl == NTL - 1 && ch_ok) {
#pragma unroll
    for (int v = 0; v < VEC; ++v) a.h_last[b * p.D + d0 + v] = carry[v];
  }
  // The last block out marks the forward complete (for the backward's check).
  __syncthreads();
  if (threadIdx.x == 0) {
    FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
    __threadfence();
    if (atomicAdd(&fh->exited, 1u) == gridDim.x - 1) {
      fh->tag = p.tag;
      __threadfence();
      fh->complete = 1u;
    }
  }
}

// ----------------------------------------------------------------- backward

template <typename T, class M, int NVL>
__global__ void __launch_bounds__(128) chain_bwd_kernel(const ChainBwdArgs a) {
  using IO = Io<T, 4>;
  using Raw = typename IO::Raw;
  constexpr int VEC = 4;
  constexpr int NTL = 32 / NVL;
  constexpr int CH = NVL * VEC;
  constexpr int BS = NTL * kTc;
  const Plan& p = a.p;
  __shared__ int s_flag;
  FwdHeader* fh = reinterpret_cast<FwdHeader*>(a.ws + p.off_fhdr);
  BwdHeader* bh = reinterpret_cast<BwdHeader*>(a.ws + p.off_bhdr);
  if (threadIdx.x == 0) {
    const bool ok = __ldcg(&fh->tag) == p.tag && __ldcg(&fh->complete) == 1u;
    if (!ok) atomicOr(&fh->err, kErrWorkspace);
    s_flag = ok;
  }
  __syncthreads();
  if (!s_flag) return;  // no forward carries for this problem: write nothing

  const int lane = threadIdx.x & 31;
  const int64_t wid = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t n_cg = (p.D + CH - 1) / CH;
  const bool warp_ok = wid < p.B * n_cg;
  const int64_t b = warp_ok ? wid / n_cg : 0;
  const int64_t d0 = warp_ok ? (wid - b * n_cg) * CH + (lane % NVL) * VEC : p.D;
  const int tcl = lane / NVL;
  const bool ch_ok = d0 < p.D;
  const int64_t BD = p.B * p.D;
  const T* x = static_cast<const T*>(a.x);
  const T* gl = static_cast<const T*>(a.gl);
  const T* dh = static_cast<const T*>(a.dh);
  T* dx = static_cast<T*>(a.dx);
  T* dgl = static_cast<T*>(a.dgl);
  const float* fpre = reinterpret_cast<const float*>(a.ws + p.off_fpre);
  const float* kd = reinterpret_cast<const float*>(a.ws + p.off_k);
  double* dlam_acc = reinterpret_cast<double*>(a.ws + p.off_dlam);

  float k[VEC], wc[VEC], dlr[VEC];
#pragma unroll
  for (int v = 0; v < VEC; ++v) {
    k[v] = 0.0f;
    wc[v] = 0.0f;
    dlr[v] = 0.0f;
  }
  if (ch_ok) {
    load_f32<VEC>(kd + d0, k);
    if (a.dh_last != nullptr) load_f32<VEC>(a.dh_last + b * p.D + d0, wc);
  }
  const int64_t nblk = (p.L + BS - 1) / BS;
  Raw rg[kTc], rx[kTc], rr[kTc], ri[kTc];
  float nhc[VEC];
  auto fetch = [&](int64_t j) {
    const int64_t t0 = j * BS + tcl * kTc;
#pragma unroll
    for (int v = 0; v < VEC; ++v) nhc[v] = 0.0f;
    if (!ch_ok) return;
    if (j > 0)
      load_f32<VEC>(fpre + (j - 1) * BD + b * p.D + d0, nhc);
    else if (a.h0 != nullptr)
      load_f32<VEC>(a.h0 + b * p.D + d0, nhc);
    const int64_t row = b * p.L + t0;
    const T* pd = dh + row * p.D + d0;
    const T* px = x + row * p.D + d0;
    const T* pg = gl + row * 2 * p.D + d0;
#pragma unroll
    for (int s = 0; s < kTc; ++s) {
      if (t0 + s < p.L) {
        rg[s] = IO::load_raw(pd + s * p.D);
        rx[s] = IO::load_raw(px + s * p.D);
        rr[s] = IO::load_raw(pg + s * 2 * p.D);
        ri[s] = IO::load_raw(pg + s * 2 * p.D + p.D);
      }
    }
  };
  if (warp_ok) fetch(nblk - 1);
  for (int64_t j = nblk - 1; warp_ok && j >= 0; --j) {
    const int64_t t0 = j * BS + tcl * kTc;
    const int64_t left = ch_ok ? p.L - t0 : 0;
    const int valid = (int)(left < 0 ? 0 : (left > kTc ? kTc : left));
    float hc[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) hc[v] = nhc[v];
    float gv[kTc][VEC], xv[kTc][VEC], ev[kTc][VEC], rv[kTc][VEC], iv[kTc][VEC];
    float A[VEC], U[VEC], W[VEC];
    if (valid == kTc)
      bwd_chunk<IO, M, true>(k, rg, rx, rr, ri, valid, gv, xv, ev, rv, iv, A, U, W);
    else
      bwd_chunk<IO, M, false>(k, rg, rx, rr, ri, valid, gv, xv, ev, rv, iv, A, U, W);
    if (j > 0) fetch(j - 1);  // the previous block's loads overlap this block
    float A2[VEC], ea[VEC], eu[VEC], sa[VEC], sw[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) A2[v] = A[v];
    chain_prefix<NVL, VEC>(A, U, tcl, ea, eu);
    chain_suffix<NVL, VEC>(A2, W, tcl, sa, sw);
    float hs[VEC], wn[VEC];
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      hs[v] = fmaf(ea[v], hc[v], eu[v]);
      wn[v] = fmaf(sa[v], wc[v], sw[v]);
    }
    // w entering the block from the later steps, for the next (earlier) block:
    // the first time lane's inclusive suffix map on this block's carry
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
      const float fa = __shfl_sync(kFull, A2[v], lane % NVL);
      const float fw = __shfl_sync(kFull, W[v], lane % NVL);
      wc[v] = fmaf(fa, wc[v], fw);
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
    const int64_t row = b * p.L + t0;
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
        float beta, uu, c2;
        M::norm_terms(q, i, xv[s][v], alpha, beta, uu, c2);
        const float dl = g * alpha * (hs[v] - c2);
        orho[v] = dl * k[v] * (r - r * r);
        oiota[v] = g * uu * (1.0f - i);
        ox[v] = g * beta;
        dlr[v] = fmaf(dl, r, dlr[v]);
        hs[v] = fmaf(alpha, hs[v], uu);
      }
      if (s < valid) {
        IO::store(pdx + s * p.D, ox);
        IO::store(pdg + s * 2 * p.D, orho);
        IO::store(pdg + s * 2 * p.D + p.D, oiota);
      }
    }
  }
  if (warp_ok) {
    if (a.dh0 != nullptr && tcl == 0 && ch_ok) {  // w at the first step
#pragma unroll
      for (int v = 0; v < VEC; ++v) a.dh0[b * p.D + d0 + v] = wc[v];
    }
    // dLambda: sum over the time lanes, one float64 add per channel
#pragma unroll
    for (int v = 0; v < VEC; ++v) {
#pragma unroll
      for (int off = 1; off < NTL; off <<= 1) dlr[v] += __shfl_down_sync(kFull, dlr[v], off * NVL);
    }
    if (tcl == 0 && ch_ok) {
      double* acc = dlam_acc + (b % kStripes) * p.D + d0;
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

}  // namespace blr
