// Device helpers of the BD-LRU kernels: vector I/O per dtype, the gate
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
// One lane moves VEC consecutive channels of one row with one access. Inputs
// are streamed (read once: evict-first), outputs are written once.

template <typename T, int VEC>
struct Io;

// Raw loads are kept packed (Raw) until they are used, so that the next tile's
// inputs can be in flight while the current tile is finished.

template <>
struct Io<float, 4> {  // 16 bytes
  using T = float;
  using Raw = float4;
  static constexpr int VEC = 4;
  static __device__ __forceinline__ Raw load_raw(const T* p) {
    return __ldcs(reinterpret_cast<const float4*>(p));
  }
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[4]) {
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[4]) {
    __stcs(reinterpret_cast<float4*>(p), make_float4(v[0], v[1], v[2], v[3]));
  }
};

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);  // round to nearest even
  return *reinterpret_cast<uint32_t*>(&b);
}

template <>
struct Io<__nv_bfloat16, 8> {  // 16 bytes
  using T = __nv_bfloat16;
  using Raw = uint4;
  static constexpr int VEC = 8;
  static __device__ __forceinline__ Raw load_raw(const T* p) {
    return __ldcs(reinterpret_cast<const uint4*>(p));
  }
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[8]) {
    v[0] = bf16_lo(t.x); v[1] = bf16_hi(t.x); v[2] = bf16_lo(t.y); v[3] = bf16_hi(t.y);
    v[4] = bf16_lo(t.z); v[5] = bf16_hi(t.z); v[6] = bf16_lo(t.w); v[7] = bf16_hi(t.w);
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[8]) {
    __stcs(reinterpret_cast<uint4*>(p), make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                                   pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7])));
  }
};

template <>
struct Io<__nv_bfloat16, 4> {  // 8 bytes
  using T = __nv_bfloat16;
  using Raw = uint2;
  static constexpr int VEC = 4;
  static __device__ __forceinline__ Raw load_raw(const T* p) {
    return __ldcs(reinterpret_cast<const uint2*>(p));
  }
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[4]) {
    v[0] = bf16_lo(t.x); v[1] = bf16_hi(t.x); v[2] = bf16_lo(t.y); v[3] = bf16_hi(t.y);
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[4]) {
    __stcs(reinterpret_cast<uint2*>(p), make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3])));
  }
};

template <int N>
__device__ __forceinline__ void load_f32(const float* p, float (&v)[N]) {
#pragma unroll
  for (int j = 0; j < N; j += 4) {
    const float4 t = *reinterpret_cast<const float4*>(p + j);
    v[j] = t.x; v[j + 1] = t.y; v[j + 2] = t.z; v[j + 3] = t.w;
  }
}

// ------------------------------------------------------------- gate arithmetic
//
// Sec. 3.2:  r = sigmoid(rho), i = sigmoid(iota), alpha = exp(-c softplus(Lambda) r),
// beta = sqrt(1 - alpha^2) i.  With k = -c softplus(Lambda) (one per channel) and
// l = k r = log(alpha) <= 0, E = expm1(l) gives both alpha = 1 + E and
// 1 - alpha^2 = -E (2 + E), without the cancellation of 1 - alpha*alpha when
// alpha is close to 1 (slow decays).
//
// Two precision policies. Float32 I/O (MathPrecise) uses CUDA's accurate expf,
// correctly rounded reciprocal, division and square root, and a degree-8
// Taylor polynomial for expm1. Bfloat16 I/O (MathFast), whose outputs carry 8
// significant bits, uses the hardware approximations: sigmoid(z) =
// (1 + tanh(z/2)) / 2 with tanh.approx (relative error below 2^-10.9),
// ex2.approx, sqrt.approx and rsqrt.approx, and a degree-5 polynomial.

__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float sqrt_approx(float x) {
  float y;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rsqrt_approx(float x) {
  float y;
  asm("rsqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Taylor polynomial of e^l - 1 = l (1 + l/2! + l^2/3! + ...) up to l^DEG / DEG!.
template <int DEG>
__device__ __forceinline__ float expm1_taylor(float l) {
  float p = 1.0f;
  float inv_fact[9] = {1.0f, 1.0f, 1.0f / 2, 1.0f / 6, 1.0f / 24, 1.0f / 120, 1.0f / 720,
                       1.0f / 5040, 1.0f / 40320};
  p = inv_fact[DEG];
#pragma unroll
  for (int j = DEG - 1; j >= 1; --j) p = fmaf(p, l, inv_fact[j]);
  return p * l;
}

struct MathPrecise {
  static __device__ __forceinline__ float sigmoid(float z) {
    return __frcp_rn(1.0f + expf(-z));
  }
  // e^l - 1 for l <= 0: the degree-8 series (truncation below l^8/9! < 5e-11
  // relative for l > -0.25) near zero, where decays usually live
  // (|l| <= softplus(Lambda) <= 0.11 for base decays in [0.9, 1)); beyond it
  // e^l < 0.78 and e^l - 1 loses nothing to cancellation.
  static __device__ __forceinline__ float expm1_nonpos(float l) {
    if (l > -0.25f) return expm1_taylor<8>(l);
    return expf(l) - 1.0f;
  }
  static __device__ __forceinline__ float sqrt(float q) { return __fsqrt_rn(q); }
  static __device__ __forceinline__ float div(float a, float b) { return __fdiv_rn(a, b); }
};

struct MathFast {
  static __device__ __forceinline__ float sigmoid(float z) {
    return fmaf(0.5f, tanh_approx(0.5f * z), 0.5f);
  }
  // Degree-5 series near zero (truncation below l^5/6! < 1.4e-6 relative for
  // l > -0.25), ex2.approx beyond.
  static __device__ __forceinline__ float expm1_nonpos(float l) {
    if (l > -0.25f) return expm1_taylor<5>(l);
    return ex2_approx(l * 1.4426950408889634f) - 1.0f;
  }
  static __device__ __forceinline__ float sqrt(float q) { return sqrt_approx(q); }
  static __device__ __forceinline__ float div(float a, float b) { return __fdividef(a, b); }
};

// k = -c softplus(Lambda), softplus(z) = max(z, 0) + log1p(exp(-|z|)), accurate.
__device__ __forceinline__ float decay_rate(float c, float lambda) {
  return -c * (fmaxf(lambda, 0.0f) + log1pf(expf(-fabsf(lambda))));
}

// ---------------------------------------------------- records and timers
//
// Look-back records are read and written with single 32- or 64-bit relaxed
// accesses at GPU scope (one access = one record, never torn; never served
// from a stale L1 line).

__device__ __forceinline__ uint32_t ld_record(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ unsigned long long ld_record(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_record(uint32_t* p, uint32_t v) {
  asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void st_record(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
// An aggregate (A, U): A in the low word (A is in [0, 1], never the empty pattern).
__device__ __forceinline__ unsigned long long pack_agg(float A, float U) {
  return (unsigned long long)__float_as_uint(A) | ((unsigned long long)__float_as_uint(U) << 32);
}
__device__ __forceinline__ bool agg_empty(unsigned long long v) { return (uint32_t)v == kEmpty; }

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Waits until the predecessor publishes its prefix or its aggregate. Returns
// false once `timeout_ns` has passed (recording kErrTimeout) or another block
// has recorded a timeout. Every path ends: the wait is bounded both by the
// global timer and by an iteration count.
__device__ __noinline__ bool wait_record(const uint32_t* pre, const unsigned long long* agg,
                                         uint32_t* err, uint64_t timeout_ns) {
  const uint64_t start = global_timer_ns();
  uint32_t sleep_ns = 32;
  for (uint32_t iter = 0;; ++iter) {
    if (ld_record(pre) != kEmpty || !agg_empty(ld_record(agg))) return true;
    __nanosleep(sleep_ns);
    if (sleep_ns < 512) sleep_ns <<= 1;
    if ((iter & 7u) == 7u) {
      if (*reinterpret_cast<volatile uint32_t*>(err) & kErrTimeout) return false;
      if (global_timer_ns() - start > timeout_ns || iter > kMaxWaitIters) {
        atomicOr(err, kErrTimeout);
        return false;
      }
    }
  }
}

// The same wait on a single flag word (the bounded-wait self-test).
__device__ __noinline__ bool wait_word(const uint32_t* flag, uint32_t* err, uint64_t timeout_ns) {
  const uint64_t start = global_timer_ns();
  uint32_t sleep_ns = 32;
  for (uint32_t iter = 0;; ++iter) {
    if (ld_record(flag) != 0u) return true;
    __nanosleep(sleep_ns);
    if (sleep_ns < 512) sleep_ns <<= 1;
    if ((iter & 7u) == 7u) {
      if (*reinterpret_cast<volatile uint32_t*>(err) & kErrTimeout) return false;
      if (global_timer_ns() - start > timeout_ns || iter > kMaxWaitIters) {
        atomicOr(err, kErrTimeout);
        return false;
      }
    }
  }
}

}  // namespace blr
