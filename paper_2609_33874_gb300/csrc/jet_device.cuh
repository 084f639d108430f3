// Device helpers shared by the kernels of libjet (header-only).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "jet.h"

namespace jet {

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

// ---- programmatic dependent launch -------------------------------------------
// Every kernel of libjet is launched with programmatic stream serialization
// (launch_pdl), so it may start while the kernel before it in the stream still
// runs. pdl_begin() lets the kernel after it start early in turn, then waits
// until all earlier work in the stream has completed and its writes are
// visible. A kernel touches no global memory before pdl_begin(); setting up
// shared memory and barriers may come first.
__device__ __forceinline__ void pdl_begin() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// record the first error a kernel meets; later ones keep the first code
__device__ __forceinline__ void flag(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// (max, sum of exp relative to max) pair combination; an empty pair is
// (-inf, 0)
__device__ __forceinline__ void ms_combine(float& m, float& s, float m2, float s2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  s = s * __expf(m - mn) + s2 * __expf(m2 - mn);
  m = mn;
}

// the same in base 2: s = sum 2^(x - m)
__device__ __forceinline__ void ms_combine2(float& m, float& s, float m2, float s2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  s = s * exp2f(m - mn) + s2 * exp2f(m2 - mn);
  m = mn;
}

}  // namespace jet
