// Device helpers of the BD-LRU kernels: 16-byte vector I/O per dtype, the gate
// arithmetic of Sec. 3.2 in float32, and the flag / timer primitives of the
// inter-block look-back.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "blr_plan.h"

namespace blr {

// ----------------------------------------------------------------- vector I/O
//
// One thread moves `kVec` consecutive channels of one row with one 16-byte
// access: 4 float32 or 8 bfloat16. Rows are contiguous along the channels, so
// the threads of a warp with consecutive tx cover whole 32-byte sectors.

struct IoF32 {
  using T = float;
  static constexpr int kVec = 4;
  static __device__ __forceinline__ void load(const T* p, float (&v)[kVec]) {
    const float4 t = *reinterpret_cast<const float4*>(p);
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[kVec]) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
};

struct IoBF16 {
  using T = __nv_bfloat16;
  static constexpr int kVec = 8;
  static __device__ __forceinline__ void load(const T* p, float (&v)[kVec]) {
    const uint4 t = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {  // bf16 -> f32 is exact: the bits move up 16 places
      v[2 * j] = __uint_as_float(w[j] << 16);
      v[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[kVec]) {
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {  // round to nearest even
      __nv_bfloat162 b = __floats2bfloat162_rn(v[2 * j], v[2 * j + 1]);
      w[j] = *reinterpret_cast<uint32_t*>(&b);
    }
    *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
  }
};

// Four float32 values of a (D)-vector, 16-byte aligned.
__device__ __forceinline__ void load_f32x4(const float* p, float* v) {
  const float4 t = *reinterpret_cast<const float4*>(p);
  v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
}

// ------------------------------------------------------------- gate arithmetic
//
// Sec. 3.2:  r = sigmoid(rho), i = sigmoid(iota), alpha = exp(-c softplus(Lambda) r),
// beta = sqrt(1 - alpha^2) i.  With k = -c softplus(Lambda) (one per channel) and
// l = k r = log(alpha) <= 0, E = expm1(l) gives both alpha = 1 + E and
// 1 - alpha^2 = -E (2 + E) without the cancellation of 1 - alpha*alpha when
// alpha is close to 1 (slow decays).
//
// Two precision policies: float32 I/O uses CUDA's accurate expf and IEEE
// division and square root; bfloat16 I/O, whose outputs carry 8 significant
// bits, uses the hardware approximations __expf, __fdividef and rsqrt.

struct MathPrecise {
  static __device__ __forceinline__ float sigmoid(float z) { return 1.0f / (1.0f + expf(-z)); }
  static __device__ __forceinline__ float exp(float l) { return expf(l); }
  static __device__ __forceinline__ float sqrt(float q) { return sqrtf(q); }
  static __device__ __forceinline__ float div(float a, float b) { return a / b; }
};

struct MathFast {
  static __device__ __forceinline__ float sigmoid(float z) {
    return __fdividef(1.0f, 1.0f + __expf(-z));
  }
  static __device__ __forceinline__ float exp(float l) { return __expf(l); }
  static __device__ __forceinline__ float sqrt(float q) { return q > 0.0f ? q * rsqrtf(q) : 0.0f; }
  static __device__ __forceinline__ float div(float a, float b) { return __fdividef(a, b); }
};

// e^l - 1 for l <= 0. Near zero (the usual range: |l| <= softplus(Lambda) <= 0.11
// for decays initialised in [0.9, 0.999]) it is the Taylor series of exp to
// degree 8, whose truncation is below l^8 / 9! < 5e-11 relative for l > -0.25;
// further out e^l - 1 loses nothing to cancellation (e^l < 0.78).
template <class M>
__device__ __forceinline__ float expm1_nonpos(float l) {
  if (l > -0.25f) {
    float p = 1.0f / 40320.0f;
    p = fmaf(p, l, 1.0f / 5040.0f);
    p = fmaf(p, l, 1.0f / 720.0f);
    p = fmaf(p, l, 1.0f / 120.0f);
    p = fmaf(p, l, 1.0f / 24.0f);
    p = fmaf(p, l, 1.0f / 6.0f);
    p = fmaf(p, l, 0.5f);
    p = fmaf(p, l, 1.0f);
    return p * l;
  }
  return M::exp(l) - 1.0f;
}

// k = -c softplus(Lambda), softplus(z) = max(z, 0) + log1p(exp(-|z|)).
__device__ __forceinline__ float decay_rate(float c, float lambda) {
  return -c * (fmaxf(lambda, 0.0f) + log1pf(expf(-fabsf(lambda))));
}

// The gates of one element: r, i, alpha and q = 1 - alpha^2 (Sec. 3.2).
template <class M>
__device__ __forceinline__ void gates(float k, float rho, float iota, float& r, float& i,
                                      float& alpha, float& q) {
  r = M::sigmoid(rho);
  i = M::sigmoid(iota);
  const float e = expm1_nonpos<M>(k * r);
  alpha = 1.0f + e;
  q = -e * (2.0f + e);
}

// ------------------------------------------------------------ flags and timers

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits until *flag != 0 and returns it, or returns 0 once `timeout_ns` has
// passed (recording kErrTimeout) or another block has recorded a timeout.
// Every path ends: the wait is bounded both by the global timer and by an
// iteration count.
__device__ __noinline__ uint32_t wait_flag(const uint32_t* flag, uint32_t* err,
                                           uint64_t timeout_ns) {
  uint32_t f = ld_acquire(flag);
  if (f != 0) return f;
  const uint64_t start = global_timer_ns();
  uint32_t sleep_ns = 32;
  for (uint32_t iter = 0;; ++iter) {
    __nanosleep(sleep_ns);
    if (sleep_ns < 512) sleep_ns <<= 1;
    f = ld_acquire(flag);
    if (f != 0) return f;
    if ((iter & 7u) == 7u) {
      if (*reinterpret_cast<volatile uint32_t*>(err) & kErrTimeout) return 0;
      if (global_timer_ns() - start > timeout_ns || iter > kMaxWaitIters) {
        atomicOr(err, kErrTimeout);
        return 0;
      }
    }
  }
}

}  // namespace blr
