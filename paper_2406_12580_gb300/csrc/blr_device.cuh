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
  // v = t / 2, halved on the packed pairs (an exponent decrement).
  static __device__ __forceinline__ void unpack_half(const Raw& t, float (&v)[4]) {
    uint32_t a, b;
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(a) : "r"(t.x), "r"(0x3f003f00u));
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(b) : "r"(t.y), "r"(0x3f003f00u));
    v[0] = bf16_lo(a); v[1] = bf16_hi(a); v[2] = bf16_lo(b); v[3] = bf16_hi(b);
  }
};

template <>
struct Io<float, 1> {  // 4 bytes
  using T = float;
  using Raw = float;
  static constexpr int VEC = 1;
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[1]) { v[0] = t; }
  static __device__ __forceinline__ void store(T* p, const float (&v)[1]) { __stcs(p, v[0]); }
  static __device__ __forceinline__ void store_smem(unsigned char* p, const float (&v)[VEC]) {
    *reinterpret_cast<float*>(p) = v[0];
  }
};

template <>
struct Io<float, 2> {  // 8 bytes
  using T = float;
  using Raw = float2;
  static constexpr int VEC = 2;
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[2]) {
    v[0] = t.x; v[1] = t.y;
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[2]) {
    __stcs(reinterpret_cast<float2*>(p), make_float2(v[0], v[1]));
  }
  static __device__ __forceinline__ void store_smem(unsigned char* p, const float (&v)[VEC]) {
    *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
  }
};

template <>
struct Io<__nv_bfloat16, 2> {  // 4 bytes
  using T = __nv_bfloat16;
  using Raw = uint32_t;
  static constexpr int VEC = 2;
  static __device__ __forceinline__ void unpack(const Raw& t, float (&v)[2]) {
    v[0] = __uint_as_float(t << 16); v[1] = __uint_as_float(t & 0xffff0000u);
  }
  static __device__ __forceinline__ void store(T* p, const float (&v)[2]) {
    __stcs(reinterpret_cast<unsigned int*>(p), pack_bf16x2(v[0], v[1]));
  }
  static __device__ __forceinline__ void store_smem(unsigned char* p, const float (&v)[VEC]) {
    *reinterpret_cast<uint32_t*>(p) = pack_bf16x2(v[0], v[1]);
  }
  // v = t / 2, halved on the packed pair (exact: an exponent decrement).
  static __device__ __forceinline__ void unpack_half(const Raw& t, float (&v)[2]) {
    uint32_t u;
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(u) : "r"(t), "r"(0x3f003f00u));  // (0.5, 0.5)
    v[0] = __uint_as_float(u << 16);
    v[1] = __uint_as_float(u & 0xffff0000u);
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
// Two precision policies, both on the hardware's approximate units (whose
// relative errors are at most about 2^-22 for ex2, rcp, rsqrt and sqrt, and
// 2^-10.9 for tanh):
//  * MathPrecise (float32 I/O): sigmoid(z) = 1 / (1 + 2^(-z log2 e)) with
//    ex2.approx and rcp.approx (relative error below ~1.5e-6 for |z| <= 10),
//    square roots through rsqrt.approx, and a degree-6 Taylor polynomial for
//    expm1. End to end this keeps the float32 outputs near 1e-6 of float64.
//  * MathFast (bfloat16 I/O, 8 significant bits out): sigmoid(z) =
//    (1 + tanh(z/2)) / 2 with tanh.approx, and a degree-4 polynomial.

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

__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// sqrt(q) and 1 / sqrt(q) for q >= 0 (0 and 0 at q = 0).
__device__ __forceinline__ void sqrt_pair(float q, float& n, float& inv_n) {
  const float rs = rsqrt_approx(q);
  const bool pos = q > 0.0f;
  n = pos ? q * rs : 0.0f;
  inv_n = pos ? rs : 0.0f;
}

struct MathPrecise {
  static __device__ __forceinline__ float sigmoid(float z) {
    return rcp_approx(1.0f + ex2_approx(-1.4426950408889634f * z));
  }
  // e^l - 1 for -0.25 < l <= 0: the degree-6 series (truncation below
  // l^6/7! < 5e-8 relative). Decays usually live there: |l| <= softplus(Lambda)
  // <= 0.11 for base decays in [0.9, 1).
  static __device__ __forceinline__ float expm1_poly(float l) { return expm1_taylor<6>(l); }
  // Any l <= 0: beyond the series' range e^l < 0.78 and e^l - 1 loses
  // nothing to cancellation.
  static __device__ __forceinline__ float expm1_any(float l) {
    if (l > -0.25f) return expm1_taylor<6>(l);
    return ex2_approx(l * 1.4426950408889634f) - 1.0f;
  }
  // sqrt(q) for q >= 0 (one sqrt.approx; 0 at q = 0, denormals flushed)
  static __device__ __forceinline__ float sqrt(float q) { return sqrt_approx(q); }
  // beta = sqrt(q) i, u = beta x and c2 = alpha u / q (= alpha i x / n).
  static __device__ __forceinline__ void norm_terms(float q, float i, float x, float alpha,
                                                    float& beta, float& u, float& c2) {
    float n, inv_n;
    sqrt_pair(q, n, inv_n);
    beta = n * i;
    u = beta * x;
    c2 = alpha * u * (inv_n * inv_n);
  }
};

struct MathFast {
  static __device__ __forceinline__ float sigmoid(float z) {
    return fmaf(0.5f, tanh_approx(0.5f * z), 0.5f);
  }
  // Degree-4 series for -0.25 < l <= 0 (truncation below l^4/5! < 3.3e-5
  // relative), ex2.approx beyond.
  static __device__ __forceinline__ float expm1_poly(float l) { return expm1_taylor<4>(l); }
  static __device__ __forceinline__ float expm1_any(float l) {
    if (l > -0.25f) return expm1_taylor<4>(l);
    return ex2_approx(l * 1.4426950408889634f) - 1.0f;
  }
  static __device__ __forceinline__ float sqrt(float q) { return sqrt_approx(q); }
  static __device__ __forceinline__ void norm_terms(float q, float i, float x, float alpha,
                                                    float& beta, float& u, float& c2) {
    float n, inv_n;
    sqrt_pair(q, n, inv_n);
    beta = n * i;
    u = beta * x;
    c2 = alpha * u * (inv_n * inv_n);
  }
};

// ------------------------------------------------- per-element gate terms
//
// The serial kernels evaluate the gates of one element with as few
// instructions as the precision policy allows. With l = k r = log(alpha) and
// E = e^l - 1 (so alpha = 1 + E and 1 - alpha^2 = -E (2 + E)):
//   decay_log(rho): l. MathFast folds sigmoid(rho) = (1 + tanh(rho/2)) / 2 into
//     l = kh tanh(rho/2) + kh with kh = k/2 (one multiply-add after tanh).
//   expm1<POLY>(l): the policy's Taylor series when every l of the channel lies
//     in (-kExpm1Series, 0] (POLY), else the series or ex2 - 1 beyond it.
constexpr float kExpm1Series = 0.25f;

template <int DEG, bool POLY>
__device__ __forceinline__ float expm1_neg(float l) {
  const float e = expm1_taylor<DEG>(l);
  if (POLY) return e;
  return l > -kExpm1Series ? e : ex2_approx(l * 1.4426950408889634f) - 1.0f;
}

// SiLU(z) = z sigmoid(z) and SiLU'(z) = sigmoid(z) (1 + z (1 - sigmoid(z))), the
// merge gate of the gated recurrent layer (Alg. 1), on the value as the policy
// unpacks it (z itself for GatesPrecise, z/2 for GatesFast).
struct GatesPrecise : MathPrecise {
  static constexpr int kDeg = 6;
  static constexpr bool kHalfInputs = false;
  static __device__ __forceinline__ float decay_log(float rho, float k, float) {
    return k * sigmoid(rho);
  }
  static __device__ __forceinline__ float silu(float z) { return z * sigmoid(z); }
  static __device__ __forceinline__ void silu_grad(float z, float& f, float& df) {
    const float sg = sigmoid(z);
    f = z * sg;
    df = fmaf(sg, z - f, sg);  // z (1 - sg) = z - f
  }
};

struct GatesFast : MathFast {
  static constexpr int kDeg = 4;
  // With rho/2, iota/2 and x/2 at hand (halved on packed bfloat16 pairs):
  // l = kh tanh(rho/2) + kh and i x = (x/2) tanh(iota/2) + x/2.
  static constexpr bool kHalfInputs = true;
  static __device__ __forceinline__ float decay_log_half(float hrho, float kh) {
    return fmaf(kh, tanh_approx(hrho), kh);
  }
  static __device__ __forceinline__ float gated_x_half(float hiota, float hx) {
    return fmaf(hx, tanh_approx(hiota), hx);
  }
  static __device__ __forceinline__ float sigmoid_half(float hz) {  // sigmoid(2 hz)
    return fmaf(0.5f, tanh_approx(hz), 0.5f);
  }
  static __device__ __forceinline__ float decay_log(float rho, float, float kh) {
    return fmaf(kh, tanh_approx(0.5f * rho), kh);
  }
  // With hz = z/2 and th = tanh(hz): SiLU = hz (1 + th), sigmoid = (1 + th)/2
  // and z (1 - sigmoid) = hz (1 - th).
  static __device__ __forceinline__ float silu(float hz) { return fmaf(hz, tanh_approx(hz), hz); }
  static __device__ __forceinline__ void silu_grad(float hz, float& f, float& df) {
    const float th = tanh_approx(hz);
    const float sg = fmaf(0.5f, th, 0.5f);
    f = fmaf(hz, th, hz);
    df = fmaf(sg, fmaf(-hz, th, hz), sg);
  }
};

template <class G>
struct GatePolicy;
template <>
struct GatePolicy<MathPrecise> {
  using type = GatesPrecise;
};
template <>
struct GatePolicy<MathFast> {
  using type = GatesFast;
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
// An aggregate (A, U): A in the low word. The tiled kernels store A in [0, 1],
// the chained forward A - 1 in (-1, 0]: a finite float, never the empty pattern.
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
  uint32_t sleep_ns = 16;
  for (uint32_t iter = 0;; ++iter) {
    if (ld_record(pre) != kEmpty || !agg_empty(ld_record(agg))) return true;
    __nanosleep(sleep_ns);
    if (sleep_ns < 128) sleep_ns <<= 1;
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

// ------------------------------------------------------------- TMA and mbarrier
//
// Tiles of the inputs are moved into shared memory by the tensor memory
// accelerator (cp.async.bulk.tensor, 3-D boxes of 32 channels x tile steps x
// one batch row) and counted on an mbarrier per pipeline stage.

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
               "r"(bytes)
               : "memory");
}

// A plain arrival (no transaction bytes): completes a phase of count 1.
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// The same test, letting the hardware suspend the thread for up to
// `hint_ns` while the phase is incomplete (instead of returning at once).
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
constexpr uint32_t kMbarSleepNs = 20000;  // per test; the whole wait stays bounded below

// Waits for the stage's loads to land. Bounded: after the limit the block
// records kErrTimeout and goes on with whatever the stage holds.
__device__ __forceinline__ void mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* err) {
  if (mbar_try_wait_sleep(bar, parity, kMbarSleepNs)) return;
  const uint64_t start = global_timer_ns();
  for (uint32_t iter = 0;; ++iter) {
    if (mbar_try_wait_sleep(bar, parity, kMbarSleepNs)) return;
    if ((iter & 15u) == 15u && (global_timer_ns() - start > kWaitTimeoutNs || iter > kMaxWaitIters)) {
      atomicOr(err, kErrTimeout);
      return;
    }
  }
}

// One 3-D tile load: box at (c0, c1, c2) of the tensor map into shared memory.
__device__ __forceinline__ void tma_load_3d(void* dst, const void* tmap, uint64_t* bar, int c0,
                                            int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_addr(dst)),
      "l"(tmap), "r"(c0), "r"(c1), "r"(c2), "r"(smem_addr(bar))
      : "memory");
}

// One 3-D tile store: shared memory into the box at (c0, c1, c2) of the tensor
// map; elements outside the tensor are not written. The writes of the box in
// shared memory must be fenced to the async proxy first.
__device__ __forceinline__ void tma_store_3d(const void* tmap, const void* src, int c0, int c1,
                                             int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(tmap),
      "r"(smem_addr(src)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Waits until at most N committed store groups still read shared memory.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// Waits until every committed store group has completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ------------------------------------------------------------ tensor memory
//
// The chained forward parks each tile's per-step states in the SM's tensor
// memory (TMEM, 128 lanes x 512 columns of 32 bits) between its two passes.
// A warp reaches only the 32 lanes of its quarter (warp index % 4) and moves
// 16 consecutive columns of its own lane per thread with one instruction.
// Addresses: lane in bits 31..16, column in bits 15..0.

// Allocates `ncols` columns (a power of two, 32..512) for the block; the
// whole warp executes it; the address is written to shared memory at `dst`.
__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tmem_fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// 16 columns of this thread's lane from 16 registers (warp-collective). The
// store completes asynchronously (tmem_wait_st).
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}
// Starts loading 16 columns of this thread's lane into 16 registers
// (warp-collective). The registers hold the data only after tmem_ld_wait on
// them: that statement names them as inputs and outputs, so no use of them can
// be scheduled before it. Stores to the same columns must have completed
// (tmem_wait_st) before the load starts.
__device__ __forceinline__ void tmem_ld16_start(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
      "%13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
                 "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]),
                 "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}
// Waits until this thread's tmem_st16 stores have completed.
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

}  // namespace blr
