// LM head with on-chip log-sum-exp partials, float32 FMA path (Eq. 1, Eq. 2).
//
// z_{n,v} = hidden[n] . w_lm[v] for a 32-row x 128-vocabulary tile; the
// tile's logits are reduced on chip to one (max, sum of exp) pair per row and
// the logits of the targets that fall in the tile are kept (Sec. 4.2: only
// the needed log-probabilities leave the GPU). float32 inputs take this path:
// the tensor cores would round them to tf32. bf16 inputs take the tcgen05
// kernel instead.
#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

constexpr int kBM = 32;        // rows per tile
constexpr int kBV = kVocabTile;  // vocabulary entries per tile (128)
constexpr int kBK = 32;        // hidden elements per step
constexpr int kThreads = 256;  // warp w owns rows 4w..4w+3; lane owns vocab lane + 32 jj

template <typename T>
__global__ void __launch_bounds__(kThreads)
lmhead_simt_kernel(const int32_t* __restrict__ target_ids, const int32_t* __restrict__ row_tgt_offset,
                   const int32_t* __restrict__ row_tgt_index, int N, int T_, int V, int D,
                   const T* __restrict__ hidden, const T* __restrict__ w_lm,
                   float2* __restrict__ part, float* __restrict__ z_tgt, int* status) {
  pdl_begin();
  __shared__ float Hs[kBK][kBM + 1];
  __shared__ float Ws[kBK][kBV + 1];
  const int row0 = blockIdx.x * kBM;
  const int vt = blockIdx.y;
  const int v0 = vt * kBV;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

  for (int k0 = 0; k0 < D; k0 += kBK) {
    __syncthreads();
    for (int i = tid; i < kBM * kBK; i += kThreads) {
      const int rr = i / kBK, kk = i % kBK;
      const int n = row0 + rr, kx = k0 + kk;
      Hs[kk][rr] = (n < N && kx < D) ? to_f32(hidden[size_t(n) * D + kx]) : 0.f;
    }
    for (int i = tid; i < kBV * kBK; i += kThreads) {
      const int vv = i / kBK, kk = i % kBK;
      const int v = v0 + vv, kx = k0 + kk;
      Ws[kk][vv] = (v < V && kx < D) ? to_f32(w_lm[size_t(v) * D + kx]) : 0.f;
    }
    __syncthreads();
#pragma unroll 4
    for (int kk = 0; kk < kBK; ++kk) {
      float hv[4], wv[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) hv[a] = Hs[kk][4 * warp + a];
#pragma unroll
      for (int b = 0; b < 4; ++b) wv[b] = Ws[kk][lane + 32 * b];
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(hv[a], wv[b], acc[a][b]);
    }
  }

  // epilogue: per row, base-2 (max, sum) over the tile's vocabulary, target gather
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int n = row0 + 4 * warp + a;
    constexpr float kLog2e = 1.4426950408889634f;
    float mx = -INFINITY;
#pragma unroll
    for (int b = 0; b < 4; ++b)
      if (v0 + lane + 32 * b < V) mx = fmaxf(mx, acc[a][b] * kLog2e);
    mx = warp_max(mx);
    float s = 0.f;
#pragma unroll
    for (int b = 0; b < 4; ++b)
      if (v0 + lane + 32 * b < V) s += exp2f(acc[a][b] * kLog2e - mx);
    s = warp_sum(s);
    if (n < N) {
      if (lane == 0) part[size_t(n) * gridDim.y + vt] = make_float2(mx, s);
      const int t0 = row_tgt_offset[n], t1 = row_tgt_offset[n + 1];
      for (int t = t0; t < t1; ++t) {
        const int j = row_tgt_index[t];
        if (j < 0 || j >= T_) {
          if (lane == 0) flag(status, JET_ERR_DEVICE);
          continue;
        }
        const int off = target_ids[j] - v0;
        if (off >= 0 && off < kBV && (off & 31) == lane) {
          const int b = off >> 5;
          z_tgt[j] = b == 0 ? acc[a][0] : b == 1 ? acc[a][1] : b == 2 ? acc[a][2] : acc[a][3];
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_lmhead_simt(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                               const void* hidden, const void* w_lm, void* ws, int* status,
                               cudaStream_t st) {
  const jet_sizes& n = lay.n;
  char* base = static_cast<char*>(ws);
  float2* part = reinterpret_cast<float2*>(base + plan.part_off);
  float* z_tgt = reinterpret_cast<float*>(base + plan.ztgt_off);
  dim3 grid(unsigned((n.N + kBM - 1) / kBM), unsigned(plan.vtiles));
  if (d.dtype == JET_DTYPE_F32) {
    return launch_pdl(lmhead_simt_kernel<float>, grid, dim3(kThreads), 0, st, lay.target_ids,
                      lay.row_tgt_offset, lay.row_tgt_index, n.N, n.T, n.V, d.D,
                      static_cast<const float*>(hidden), static_cast<const float*>(w_lm), part,
                      z_tgt, status);
  }
  return launch_pdl(lmhead_simt_kernel<__nv_bfloat16>, grid, dim3(kThreads), 0, st,
                    lay.target_ids, lay.row_tgt_offset, lay.row_tgt_index, n.N, n.T, n.V, d.D,
                    static_cast<const __nv_bfloat16*>(hidden),
                    static_cast<const __nv_bfloat16*>(w_lm), part, z_tgt, status);
}

}  // namespace jet
