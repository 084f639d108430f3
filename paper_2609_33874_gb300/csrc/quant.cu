// Per-row e4m3 quantisation for the low-precision LM head (Appendix A: the
// paper's models run with 8-bit and 4-bit weights). A row x of bf16 values
// becomes OCP FP8 E4M3 codes q and one float32 scale s with x ~= s decode(q):
// amax = max |x| (float32), s = amax / 448, q = e4m3(x * (448 / amax)) rounded
// to nearest even and saturated at +-448 (448 is the largest e4m3 value). A
// row of zeros gets s = 0 and zero codes.
//
// The 4-bit weights (w4; the paper's largest models use 4-bit weights in
// scaled 32-element blocks, Appendix A) keep one float32 scale per row and, per
// 32-element block, a power-of-two exponent e in [-5, 0] over OCP FP4 E2M1
// codes: s = amax / 6, inv = 6 / amax, t = blockmax * inv, e = the smallest
// value in [-5, 0] with t <= 6 * 2^e (0 if none), code = e2m1(x * (inv * 2^-e))
// rounded to nearest even and saturated at +-6. They are written as the
// block-scaled LM head reads them (include/jet.h): a row-major region of
// packed codes, then one 512-byte chunk of UE8M0 factors 127 + e per
// (128-row tile, 128-code slice).
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

// E2M1 code of a float32 value: nearest of 0, .5, 1, 1.5, 2, 3, 4, 6, ties to
// the even code (each comparison is with the midpoint to the next magnitude,
// strict where the lower code is the even one), saturating, sign in bit 3
__device__ __forceinline__ uint32_t e2m1_code(float y) {
  const float a = fabsf(y);
  const uint32_t c = uint32_t(a > 0.25f) + uint32_t(a >= 0.75f) + uint32_t(a > 1.25f) +
                     uint32_t(a >= 1.75f) + uint32_t(a > 2.5f) + uint32_t(a >= 3.5f) +
                     uint32_t(a > 5.0f);
  return c | ((__float_as_uint(y) >> 28) & 8u);
}

// one warp per (padded) vocabulary row; rows past V are written as zeros
__global__ void __launch_bounds__(32 * kRowsPerBlock)
quantize_w4_kernel(const __nv_bfloat16* __restrict__ x, int V, int D, int rows_pad, int nkb,
                   uint8_t* __restrict__ w4, float* __restrict__ scale) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int v = blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (v >= rows_pad) return;
  const bool real = v < V;
  const __nv_bfloat16* xr = x + size_t(real ? v : 0) * D;
  float amax = 0.f;
  if (real) {
    for (int k = lane * 8; k < D; k += 256) {
      const uint4 q = *reinterpret_cast<const uint4*>(xr + k);
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h[i]);
        amax = fmaxf(amax, fmaxf(fabsf(f.x), fabsf(f.y)));
      }
    }
    amax = warp_max(amax);
    if (lane == 0) scale[v] = amax > 0.f ? __fdiv_rn(amax, 6.f) : 0.f;
  }
  const float inv = amax > 0.f ? __fdiv_rn(6.f, amax) : 0.f;
  const int r = v & (kVocabTile - 1), vt = v / kVocabTile;
  const int c = lane >> 3;  // the 32-element block of the slice
  const size_t sf_off = size_t(rows_pad) * nkb * 64;  // the scale factors follow the codes
  for (int kb = 0; kb < nkb; ++kb) {
    const int k = kb * 128 + lane * 4;
    float f[4] = {0.f, 0.f, 0.f, 0.f};
    if (real && k < D) {
      const uint2 q = *reinterpret_cast<const uint2*>(xr + k);
      const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.x));
      const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.y));
      f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
    }
    float bmax = fmaxf(fmaxf(fabsf(f[0]), fabsf(f[1])), fmaxf(fabsf(f[2]), fabsf(f[3])));
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) bmax = fmaxf(bmax, __shfl_xor_sync(0xffffffffu, bmax, o));
    const float t = __fmul_rn(bmax, inv);
    int e = 0;
    float thr = 6.f;  // 6 * 2^ee, exact
#pragma unroll
    for (int ee = 0; ee >= -5; --ee, thr *= 0.5f)
      if (t <= thr) e = ee;
    const float inv_b = __fmul_rn(inv, __int_as_float((127 - e) << 23));  // inv * 2^-e, exact
    // four codes, element 2 j in the low nibble of byte j
    uint32_t code = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) code |= e2m1_code(__fmul_rn(f[i], inv_b)) << (4 * i);
    *reinterpret_cast<uint16_t*>(w4 + size_t(v) * (nkb * 64) + kb * 64 + 2 * lane) =
        uint16_t(code);
    // the block's exponent as a UE8M0 scale factor, in the order one
    // tcgen05.cp (32 x 128 bits) brings a 512-byte chunk into TMEM: row
    // 32 j + i of the tile, block c of the slice at byte 16 i + 4 j + c
    if ((lane & 7) == 0)
      w4[sf_off + (size_t(vt) * nkb + kb) * 512 + 16 * (r & 31) + 4 * (r >> 5) + c] =
          uint8_t(127 + e);
  }
}

// MXFP8 (e4m3 codes, one UE8M0 scale factor per 32-element block): one warp
// per row slot. Row slots come in groups of 128 * halves; slot rs of group g
// is matrix row g * tile_rows + rs when rs < tile_rows (and that row exists),
// padding otherwise. Per 128-element slice kb the group's scale factors form
// `halves` 512-byte chunks, chunk (g * nkb + kb) * halves + rs / 128, in the
// order one tcgen05.cp (32 x 128 bits) places a chunk in TMEM: slot
// 32 j + i of the 128 at byte 16 i + 4 j + block. Codes are written row-major
// [rows, D] for the rows that exist; padding slots get factor 127 and no codes.
// X = floor(log2(block max)) - 8 from the float's exponent field (clamped to
// -127 below), element code = e4m3(x * 2^-X), nearest even, saturating.
__global__ void __launch_bounds__(32 * kRowsPerBlock)
quantize_mx_kernel(const __nv_bfloat16* __restrict__ x, int rows, int D, int slots,
                   int tile_rows, int halves, int nkb, uint8_t* __restrict__ codes,
                   uint8_t* __restrict__ sf) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int slot = blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (slot >= slots) return;
  const int G = 128 * halves;
  const int g = slot / G, rs = slot % G;
  const int row = g * tile_rows + rs;
  const bool real = rs < tile_rows && row < rows;
  const __nv_bfloat16* xr = x + size_t(real ? row : 0) * D;
  const int r = rs & 127, c = lane >> 3;
  for (int kb = 0; kb < nkb; ++kb) {
    const int k = kb * 128 + lane * 4;
    float f[4] = {0.f, 0.f, 0.f, 0.f};
    if (real && k < D) {
      const uint2 q = *reinterpret_cast<const uint2*>(xr + k);
      const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.x));
      const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&q.y));
      f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
    }
    float bmax = fmaxf(fmaxf(fabsf(f[0]), fabsf(f[1])), fmaxf(fabsf(f[2]), fabsf(f[3])));
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) bmax = fmaxf(bmax, __shfl_xor_sync(0xffffffffu, bmax, o));
    // floor(log2(bmax)) is the exponent field minus 127 for a normal float;
    // zero and subnormal maxima clamp to X = -127
    const int ef = (__float_as_int(bmax) >> 23) & 0xFF;
    const int X = ef == 0 ? -127 : max(ef - 127 - 8, -127);
    const float scale = __int_as_float((127 - X) << 23);  // 2^-X, exact (X <= 119)
    if (real && k < D) {
      uint32_t w = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        w |= uint32_t(__nv_cvt_float_to_fp8(__fmul_rn(f[i], scale), __NV_SATFINITE, __NV_E4M3))
             << (8 * i);
      *reinterpret_cast<uint32_t*>(codes + size_t(row) * D + k) = w;
    }
    if ((lane & 7) == 0)
      sf[(size_t(g * nkb + kb) * halves + (rs >> 7)) * 512 + 16 * (r & 31) + 4 * (r >> 5) + c] =
          uint8_t(real ? X + 127 : 127);
  }
}

}  // namespace

cudaError_t launch_quantize_w4(const void* x, int V, int D, uint8_t* w4, float* scale,
                               cudaStream_t st) {
  if (V <= 0) return cudaSuccess;
  const int rows_pad = (V + kVocabTile - 1) / kVocabTile * kVocabTile;
  const int nkb = (D + 127) / 128;
  return launch_pdl(quantize_w4_kernel, dim3(unsigned(rows_pad / kRowsPerBlock)),
                    dim3(32 * kRowsPerBlock), 0, st, static_cast<const __nv_bfloat16*>(x), V, D,
                    rows_pad, nkb, w4, scale);
}

cudaError_t launch_quantize_e4m3(const void* x, int rows, int D, uint8_t* q, float* scale,
                                 cudaStream_t st) {
  if (rows <= 0) return cudaSuccess;
  return launch_pdl(quantize_e4m3_kernel, dim3(unsigned((rows + kRowsPerBlock - 1) / kRowsPerBlock)),
                    dim3(32 * kRowsPerBlock), 0, st, static_cast<const __nv_bfloat16*>(x), rows, D,
                    q, scale);
}

}  // namespace jet

namespace jet {

cudaError_t launch_quantize_mx(const void* x, int rows, int D, int slots, int tile_rows,
                               int halves, uint8_t* codes, uint8_t* sf, cudaStream_t st) {
  if (slots <= 0) return cudaSuccess;
  const int nkb = (D + 127) / 128;
  return launch_pdl(quantize_mx_kernel, dim3(unsigned((slots + kRowsPerBlock - 1) / kRowsPerBlock)),
                    dim3(32 * kRowsPerBlock), 0, st, static_cast<const __nv_bfloat16*>(x), rows, D,
                    slots, tile_rows, halves, nkb, codes, sf);
}

}  // namespace jet
