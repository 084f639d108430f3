// Per-row e4m3 quantisation for the low-precision LM head (Appendix A: the
// paper's models run with 8-bit and 4-bit weights). A row x of bf16 values
// becomes OCP FP8 E4M3 codes q and one float32 scale s with x ~= s decode(q):
// amax = max |x| (float32), s = amax / 448, q = e4m3(x * (448 / amax)) rounded
// to nearest even and saturated at +-448 (448 is the largest e4m3 value). A
// row of zeros gets s = 0 and zero codes.
#include <cuda_fp8.h>

#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

constexpr int kRowsPerBlock = 8;  // one warp per row

__global__ void __launch_bounds__(32 * kRowsPerBlock)
quantize_e4m3_kernel(const __nv_bfloat16* __restrict__ x, int rows, int D,
                     uint8_t* __restrict__ q, float* __restrict__ scale) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (row >= rows) return;
  const __nv_bfloat16* xr = x + size_t(row) * D;
  float amax = 0.f;
  for (int k = lane * 8; k < D; k += 256) {
    const uint4 v = *reinterpret_cast<const uint4*>(xr + k);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(h[i]);
      amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
    }
  }
  amax = warp_max(amax);
  const float inv = amax > 0.f ? 448.f / amax : 0.f;
  if (lane == 0) scale[row] = amax / 448.f;
  uint8_t* qr = q + size_t(row) * D;
  for (int k = lane * 8; k < D; k += 256) {
    const uint4 v = *reinterpret_cast<const uint4*>(xr + k);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
    uint32_t w[2] = {0u, 0u};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(h[i]);
      const uint32_t c0 = __nv_cvt_float_to_fp8(f.x * inv, __NV_SATFINITE, __NV_E4M3);
      const uint32_t c1 = __nv_cvt_float_to_fp8(f.y * inv, __NV_SATFINITE, __NV_E4M3);
      w[i >> 1] |= (c0 | (c1 << 8)) << (16 * (i & 1));
    }
    *reinterpret_cast<uint2*>(qr + k) = make_uint2(w[0], w[1]);
  }
}

}  // namespace

cudaError_t launch_quantize_e4m3(const void* x, int rows, int D, uint8_t* q, float* scale,
                                 cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  return launch_pdl(quantize_e4m3_kernel, dim3(unsigned((rows + kRowsPerBlock - 1) / kRowsPerBlock)),
                    dim3(32 * kRowsPerBlock), 0, st, static_cast<const __nv_bfloat16*>(x), rows, D,
                    q, scale);
}

}  // namespace jet
