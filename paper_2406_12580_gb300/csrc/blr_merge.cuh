// The merge of the gated recurrent layer (Alg. 1: H'_y = H_y (x) SiLU(H_z)) as
// stand-alone elementwise kernels. Problems served by the serial kernels get
// the merge fused into the scan; the tiled look-back kernels have no fused
// form, so their gated entry points run the scan and these kernels around it,
// in place in the caller's buffers:
//   forward:  y <- y SiLU(z), where the scan left h in y;
//   backward: dh <- dy SiLU(z) (into the dx buffer, which the scan's backward
//             then reads as dh and overwrites with dx) and dz <- dy h SiLU'(z),
//             where a forward recompute left h in the dz buffer.
// Every thread handles 16-byte vectors (4 float32 or 8 bfloat16 values;
// B L D is a multiple of 8), grid-stride.
#pragma once

#include "blr_device.cuh"

namespace blr {

template <typename T>
struct MergeVec;
template <>
struct MergeVec<float> {
  using IO = Io<float, 4>;
};
template <>
struct MergeVec<__nv_bfloat16> {
  using IO = Io<__nv_bfloat16, 8>;
};

template <typename T>
__global__ void __launch_bounds__(256) merge_fwd_kernel(T* y, const T* z, int64_t n_vec) {
  using IO = typename MergeVec<T>::IO;
  constexpr int V = IO::VEC;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_vec;
       i += (int64_t)gridDim.x * blockDim.x) {
    float hv[V], zv[V], out[V];
    IO::unpack(IO::load_raw(y + i * V), hv);
    IO::unpack(IO::load_raw(z + i * V), zv);
#pragma unroll
    for (int v = 0; v < V; ++v) out[v] = hv[v] * GatesPrecise::silu(zv[v]);
    IO::store(y + i * V, out);
  }
}

template <typename T>
__global__ void __launch_bounds__(256) merge_bwd_kernel(const T* dy, const T* z, T* dh, T* hz,
                                                        int64_t n_vec) {
  using IO = typename MergeVec<T>::IO;
  constexpr int V = IO::VEC;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_vec;
       i += (int64_t)gridDim.x * blockDim.x) {
    float dyv[V], zv[V], hv[V], odh[V], odz[V];
    IO::unpack(IO::load_raw(dy + i * V), dyv);
    IO::unpack(IO::load_raw(z + i * V), zv);
    IO::unpack(IO::load_raw(hz + i * V), hv);
#pragma unroll
    for (int v = 0; v < V; ++v) {
      float f, df;
      GatesPrecise::silu_grad(zv[v], f, df);
      odh[v] = dyv[v] * f;
      odz[v] = (dyv[v] * hv[v]) * df;
    }
    IO::store(dh + i * V, odh);
    IO::store(hz + i * V, odz);
  }
}

}  // namespace blr
