// Small kernels of a decoder stack over the scoring step's rows: RMSNorm, the
// split of a full-attention layer's q/k/v projection into the step's query and
// candidate key/value buffers, the linear-attention layer's gates (per-head
// key normalisation, sigmoid decay and write strengths). The projections
// themselves run on the tensor cores (proj_tc.cu), the attention and the fork
// (which also reads the shared rows' outputs off the prefix states) on the
// step's kernels.
#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// h[n] = x[n] / sqrt(mean(x[n]^2) + eps) * g, one 512-thread block per row
// (D % 8 == 0): a row of a few KB gets sixteen warps' loads in flight; the
// fused residual-and-norm pass of the projections keeps the same order
constexpr int kNormThreads = 512;
__global__ void __launch_bounds__(kNormThreads)
rmsnorm_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ g, int N,
               int D, float eps, __nv_bfloat16* __restrict__ h) {
  pdl_begin();
  __shared__ float part[kNormThreads / 32];
  const int n = blockIdx.x, tid = threadIdx.x;
  if (n >= N) return;
  const __nv_bfloat16* xr = x + size_t(n) * D;
  float ss = 0.f;
  for (int k = tid * 8; k < D; k += kNormThreads * 8) {
    const uint4 v = *reinterpret_cast<const uint4*>(xr + k);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(p[i]);
      ss = fmaf(f.x, f.x, fmaf(f.y, f.y, ss));
    }
  }
  ss = warp_sum(ss);
  if ((tid & 31) == 0) part[tid >> 5] = ss;
  __syncthreads();
  ss = 0.f;
#pragma unroll
  for (int w = 0; w < kNormThreads / 32; ++w) ss += part[w];
  const float inv = 1.f / sqrtf(ss / float(D) + eps);
  __nv_bfloat16* hr = h + size_t(n) * D;
  for (int k = tid * 8; k < D; k += kNormThreads * 8) {
    const uint4 v = *reinterpret_cast<const uint4*>(xr + k);
    const uint4 gv = *reinterpret_cast<const uint4*>(g + k);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
    const __nv_bfloat162* pg = reinterpret_cast<const __nv_bfloat162*>(&gv);
    uint4 out;
    __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&out);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(p[i]), gg = __bfloat1622float2(pg[i]);
      po[i] = __floats2bfloat162_rn(f.x * inv * gg.x, f.y * inv * gg.y);
    }
    *reinterpret_cast<uint4*>(hr + k) = out;
  }
}

// z [N, (Hq + 2 Hkv) d] -> q [N, Hq d] (every row) and k_cand, v_cand
// [F, Hkv d] (the fed rows, fed-token index n - req - 1); one block per row,
// 16-byte pieces
__global__ void split_qkv_kernel(const __nv_bfloat16* __restrict__ z, const int32_t* row_req,
                                 const int32_t* row_cand, int N, int R, int qw, int kw,
                                 __nv_bfloat16* __restrict__ q,
                                 __nv_bfloat16* __restrict__ kc, __nv_bfloat16* __restrict__ vc,
                                 int* status) {
  pdl_begin();
  const int n = blockIdx.x;
  if (n >= N) return;
  const int r = row_req[n];
  const int zw = qw + 2 * kw;
  const uint4* zr = reinterpret_cast<const uint4*>(z + size_t(n) * zw);
  uint4* qr = reinterpret_cast<uint4*>(q + size_t(n) * qw);
  for (int e = threadIdx.x; e < qw / 8; e += blockDim.x) qr[e] = zr[e];
  if (r < 0 || r >= R) {
    if (threadIdx.x == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  // a shared row's key and value are the prefix's last position
  if (row_cand[n] < 0) return;
  const int f = n - r - 1;
  if (f < 0 || f >= N - R) {
    if (threadIdx.x == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  uint4* kr = reinterpret_cast<uint4*>(kc + size_t(f) * kw);
  uint4* vr = reinterpret_cast<uint4*>(vc + size_t(f) * kw);
  for (int e = threadIdx.x; e < kw / 8; e += blockDim.x) {
    kr[e] = zr[qw / 8 + e];
    vr[e] = zr[(qw + kw) / 8 + e];
  }
}

// z [N, Hl (2 dk + dv) + 2 Hl] -> lq_all [N, Hl, dk] (every row) and, for the
// fed rows, lq, lk (normalised per head), lv, alpha = sigmoid(a),
// beta = sigmoid(b); one warp per (row, head), dk = 128
__global__ void __launch_bounds__(256)
gates_kernel(const __nv_bfloat16* __restrict__ z, const int32_t* row_req,
             const int32_t* row_cand, int N, int R, int Hl,
             int dv, __nv_bfloat16* __restrict__ lq_all, __nv_bfloat16* __restrict__ lq,
             __nv_bfloat16* __restrict__ lk, __nv_bfloat16* __restrict__ lv,
             float* __restrict__ alpha, float* __restrict__ beta, int* status) {
  pdl_begin();
  constexpr int dk = 128;
  const int lane = threadIdx.x & 31;
  const int wid = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (wid >= N * Hl) return;
  const int n = wid / Hl, hh = wid % Hl;
  const int zw = Hl * (2 * dk + dv) + 2 * Hl;
  const __nv_bfloat16* zr = z + size_t(n) * zw;
  // this lane's 4 elements of q and k
  const uint2 qv = *reinterpret_cast<const uint2*>(zr + hh * dk + 4 * lane);
  const uint2 kv = *reinterpret_cast<const uint2*>(zr + Hl * dk + hh * dk + 4 * lane);
  *reinterpret_cast<uint2*>(lq_all + (size_t(n) * Hl + hh) * dk + 4 * lane) = qv;
  const int r = row_req[n];
  if (r < 0 || r >= R) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  if (row_cand[n] < 0) return;  // the shared row only reads the prefix state
  const int f = n - r - 1;
  if (f < 0 || f >= N - R) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  *reinterpret_cast<uint2*>(lq + (size_t(f) * Hl + hh) * dk + 4 * lane) = qv;
  const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kv.x));
  const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kv.y));
  float ss = k01.x * k01.x + k01.y * k01.y + k23.x * k23.x + k23.y * k23.y;
  ss = warp_sum(ss);
  const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
  uint2 kn;
  *reinterpret_cast<__nv_bfloat162*>(&kn.x) = __floats2bfloat162_rn(k01.x * inv, k01.y * inv);
  *reinterpret_cast<__nv_bfloat162*>(&kn.y) = __floats2bfloat162_rn(k23.x * inv, k23.y * inv);
  *reinterpret_cast<uint2*>(lk + (size_t(f) * Hl + hh) * dk + 4 * lane) = kn;
  const __nv_bfloat16* vsrc = zr + 2 * Hl * dk + hh * dv;
  __nv_bfloat16* vdst = lv + (size_t(f) * Hl + hh) * dv;
  for (int j = lane; j < dv; j += 32) vdst[j] = vsrc[j];
  if (lane == 0) {
    const float a = __bfloat162float(zr[Hl * (2 * dk + dv) + hh]);
    const float b = __bfloat162float(zr[Hl * (2 * dk + dv) + Hl + hh]);
    alpha[size_t(f) * Hl + hh] = 1.f / (1.f + expf(-a));
    beta[size_t(f) * Hl + hh] = 1.f / (1.f + expf(-b));
  }
}

// The full-attention layer's q/k/v projection, split over K, reduced straight
// into q (every row) and the fed rows' k and v: one 512-thread block per row,
// 8 columns a thread at a time, each summed over the partials
// part[splits][N][qw + 2 kw] in split order and rounded to bf16 as a stored z
// would be (the same results as the reduce and split_qkv_kernel).
__global__ void __launch_bounds__(512)
reduce_qkv_kernel(const float* __restrict__ part, int splits, const int32_t* row_req,
                  const int32_t* row_cand, int N, int R, int qw, int kw,
                  __nv_bfloat16* __restrict__ q, __nv_bfloat16* __restrict__ kc,
                  __nv_bfloat16* __restrict__ vc, int* status) {
  pdl_begin();
  const int n = blockIdx.x;
  if (n >= N) return;
  const int r = row_req[n];
  if (r < 0 || r >= R) {
    if (threadIdx.x == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  const bool fed = row_cand[n] >= 0;  // a shared row's key and value are the prefix's
  const int f = n - r - 1;
  if (fed && (f < 0 || f >= N - R)) {
    if (threadIdx.x == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  const int zw = qw + 2 * kw;
  const int pieces = fed ? zw / 8 : qw / 8;
  for (int e = threadIdx.x; e < pieces; e += blockDim.x) {
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
#pragma unroll 4
    for (int sp = 0; sp < splits; ++sp) {
      const float4* pp = reinterpret_cast<const float4*>(part + (size_t(sp) * N + n) * zw + 8 * e);
      const float4 a0 = pp[0], a1 = pp[1];
      acc[0] += a0.x; acc[1] += a0.y; acc[2] += a0.z; acc[3] += a0.w;
      acc[4] += a1.x; acc[5] += a1.y; acc[6] += a1.z; acc[7] += a1.w;
    }
    uint4 o;
    __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&o);
#pragma unroll
    for (int i = 0; i < 4; ++i) po[i] = __floats2bfloat162_rn(acc[2 * i], acc[2 * i + 1]);
    const int c = 8 * e;
    if (c < qw)
      *reinterpret_cast<uint4*>(q + size_t(n) * qw + c) = o;
    else if (c < qw + kw)
      *reinterpret_cast<uint4*>(kc + size_t(f) * kw + (c - qw)) = o;
    else
      *reinterpret_cast<uint4*>(vc + size_t(f) * kw + (c - qw - kw)) = o;
  }
}

// The linear layer's mixer projection, split over K, reduced straight into
// the gates: one warp per (row, head) sums its q, k, v and gate columns of the
// f32 partials part[splits][N][zw] in split order, rounds each to bf16 as a
// stored z would be, then does what gates_kernel does with z (the same
// results without the z round trip and its reduce pass).
__global__ void __launch_bounds__(256)
reduce_gates_kernel(const float* __restrict__ part, int splits, const int32_t* row_req,
                    const int32_t* row_cand, int N, int R, int Hl, int dv,
                    __nv_bfloat16* __restrict__ lq_all, __nv_bfloat16* __restrict__ lq,
                    __nv_bfloat16* __restrict__ lk, __nv_bfloat16* __restrict__ lv,
                    float* __restrict__ alpha, float* __restrict__ beta, int* status) {
  pdl_begin();
  constexpr int dk = 128;
  const int lane = threadIdx.x & 31;
  const int wid = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (wid >= N * Hl) return;
  const int n = wid / Hl, hh = wid % Hl;
  const int zw = Hl * (2 * dk + dv) + 2 * Hl;
  // four consecutive columns summed over the splits, rounded to bf16
  auto sum4 = [&](int col) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int sp = 0; sp < splits; ++sp) {
      const float4 x = *reinterpret_cast<const float4*>(part + (size_t(sp) * N + n) * zw + col);
      acc.x += x.x; acc.y += x.y; acc.z += x.z; acc.w += x.w;
    }
    uint2 r;
    *reinterpret_cast<__nv_bfloat162*>(&r.x) = __floats2bfloat162_rn(acc.x, acc.y);
    *reinterpret_cast<__nv_bfloat162*>(&r.y) = __floats2bfloat162_rn(acc.z, acc.w);
    return r;
  };
  auto sum1 = [&](int col) {
    float acc = 0.f;
    for (int sp = 0; sp < splits; ++sp) acc += part[(size_t(sp) * N + n) * zw + col];
    return __float2bfloat16_rn(acc);
  };
  const uint2 qv = sum4(hh * dk + 4 * lane);
  *reinterpret_cast<uint2*>(lq_all + (size_t(n) * Hl + hh) * dk + 4 * lane) = qv;
  const int r = row_req[n];
  if (r < 0 || r >= R) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  if (row_cand[n] < 0) return;  // the shared row only reads the prefix state
  const int f = n - r - 1;
  if (f < 0 || f >= N - R) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  *reinterpret_cast<uint2*>(lq + (size_t(f) * Hl + hh) * dk + 4 * lane) = qv;
  const uint2 kv = sum4(Hl * dk + hh * dk + 4 * lane);
  const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kv.x));
  const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kv.y));
  float ss = k01.x * k01.x + k01.y * k01.y + k23.x * k23.x + k23.y * k23.y;
  ss = warp_sum(ss);
  const float inv = ss > 0.f ? 1.f / sqrtf(ss) : 0.f;
  uint2 kn;
  *reinterpret_cast<__nv_bfloat162*>(&kn.x) = __floats2bfloat162_rn(k01.x * inv, k01.y * inv);
  *reinterpret_cast<__nv_bfloat162*>(&kn.y) = __floats2bfloat162_rn(k23.x * inv, k23.y * inv);
  *reinterpret_cast<uint2*>(lk + (size_t(f) * Hl + hh) * dk + 4 * lane) = kn;
  __nv_bfloat16* vdst = lv + (size_t(f) * Hl + hh) * dv;
  for (int j = lane; j < dv; j += 32) vdst[j] = sum1(2 * Hl * dk + hh * dv + j);
  if (lane == 0) {
    const float a = __bfloat162float(sum1(Hl * (2 * dk + dv) + hh));
    const float b = __bfloat162float(sum1(Hl * (2 * dk + dv) + Hl + hh));
    alpha[size_t(f) * Hl + hh] = 1.f / (1.f + expf(-a));
    beta[size_t(f) * Hl + hh] = 1.f / (1.f + expf(-b));
  }
}

}  // namespace

cudaError_t launch_reduce_qkv(const jet_layout& lay, const float* part, int splits, int qw,
                              int kw, void* q, void* kc, void* vc, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  if (n.N <= 0) return cudaSuccess;
  return launch_pdl(reduce_qkv_kernel, dim3(unsigned(n.N)), dim3(512), 0, st, part, splits,
                    lay.row_req, lay.row_cand, n.N, n.R, qw, kw, static_cast<__nv_bfloat16*>(q),
                    static_cast<__nv_bfloat16*>(kc), static_cast<__nv_bfloat16*>(vc), status);
}

cudaError_t launch_reduce_gates(const jet_layout& lay, const float* part, int splits, int Hl,
                                int dv, void* lq_all, void* lq, void* lk, void* lv,
                                float* alpha, float* beta, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  if (n.N <= 0) return cudaSuccess;
  const int warps = n.N * Hl;
  return launch_pdl(reduce_gates_kernel, dim3(unsigned((warps + 7) / 8)), dim3(256), 0, st, part,
                    splits, lay.row_req, lay.row_cand, n.N, n.R, Hl, dv,
                    static_cast<__nv_bfloat16*>(lq_all), static_cast<__nv_bfloat16*>(lq),
                    static_cast<__nv_bfloat16*>(lk), static_cast<__nv_bfloat16*>(lv), alpha, beta,
                    status);
}

cudaError_t launch_rmsnorm(const void* x, const void* g, int N, int D, float eps, void* h,
                           cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  return launch_pdl(rmsnorm_kernel, dim3(unsigned(N)), dim3(kNormThreads), 0, st,
                    static_cast<const __nv_bfloat16*>(x),
                    static_cast<const __nv_bfloat16*>(g), N, D, eps,
                    static_cast<__nv_bfloat16*>(h));
}

cudaError_t launch_split_qkv(const jet_layout& lay, const void* z, int qw, int kw, void* q,
                             void* kc, void* vc, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  if (n.N <= 0) return cudaSuccess;
  return launch_pdl(split_qkv_kernel, dim3(unsigned(n.N)), dim3(128), 0, st,
                    static_cast<const __nv_bfloat16*>(z), lay.row_req, lay.row_cand, n.N, n.R, qw,
                    kw,
                    static_cast<__nv_bfloat16*>(q), static_cast<__nv_bfloat16*>(kc),
                    static_cast<__nv_bfloat16*>(vc), status);
}

cudaError_t launch_gates(const jet_layout& lay, const void* z, int Hl, int dv, void* lq_all,
                         void* lq, void* lk, void* lv, float* alpha, float* beta, int* status,
                         cudaStream_t st) {
  const jet_sizes& n = lay.n;
  if (n.N <= 0) return cudaSuccess;
  const int warps = n.N * Hl;
  return launch_pdl(gates_kernel, dim3(unsigned((warps + 7) / 8)), dim3(256), 0, st,
                    static_cast<const __nv_bfloat16*>(z), lay.row_req, lay.row_cand, n.N, n.R, Hl,
                    dv,
                    static_cast<__nv_bfloat16*>(lq_all), static_cast<__nv_bfloat16*>(lq),
                    static_cast<__nv_bfloat16*>(lk), static_cast<__nv_bfloat16*>(lv), alpha, beta,
                    status);
}

}  // namespace jet
