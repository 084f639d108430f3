// Shared-prefix cascade attention (Sec. 4.1, Fig. 1 "KV-cache text models"):
// float32 prefix kernel, and the merge kernel shared with the bf16
// tensor-core prefix kernel (attend_tc.cu). Partials are in base 2:
// m = max of score log2(e), l = sum of 2^(score log2(e) - m).
//
// Every row of request r attends to the request's P_r prefix keys; a row fed
// with y_{c,t} additionally attends to y_{c,1..t} of its own candidate. The
// prefix part is identical for all of the request's rows, so it is computed
// per (request, key/value head) with all n_r * g query vectors of the group
// sharing each prefix K/V tile (g = Hq / Hkv): the tile is read from memory
// once per group, not once per candidate. Long prefixes are split into
// chunks; each chunk leaves an unnormalised partial (max, sum of exp, sum of
// exp-weighted values) that the merge kernel combines with the short causal
// candidate part by the usual log-sum-exp rescaling.
#include <algorithm>

#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

constexpr int kQV = 16;       // query vectors per CTA
constexpr int kKT = 32;       // keys per tile
constexpr int kThreads = 256;
constexpr long long kTargetCtas = 608;  // about four CTAs per SM on 152 SMs
constexpr int kPlanSMs = 152;           // GB300
constexpr int kMinChunkTc = 640;        // keys

template <int DH>
constexpr size_t prefix_smem_bytes() {
  return sizeof(float) * (size_t(kQV) * (DH + 1) + size_t(kKT) * (DH + 1) + size_t(kKT) * DH +
                          size_t(kQV) * (kKT + 1));
}

// One CTA: one prefix chunk of one (request, key/value head) for kQV query
// vectors. Thread (vec = tid / 16, sub = tid % 16) scores keys sub and sub+16
// of each tile for its vector and accumulates output dims sub + 16 i.
template <typename T, int DH>
__global__ void __launch_bounds__(kThreads)
attend_prefix_kernel(const int32_t* __restrict__ prefix_offset, const int32_t* __restrict__ row_offset,
                     int R, int N, int total_prefix, int Hq, int Hkv, int chunk,
                     const T* __restrict__ q, const T* __restrict__ k_pre, const T* __restrict__ v_pre,
                     float* __restrict__ o_part, float2* __restrict__ ml_part, int* status) {
  pdl_begin();
  extern __shared__ float smem[];
  float* Qs = smem;                          // [kQV][DH+1], pre-scaled by 1/sqrt(d)
  float* Ks = Qs + kQV * (DH + 1);           // [kKT][DH+1]
  float* Vs = Ks + kKT * (DH + 1);           // [kKT][DH]
  float* Ps = Vs + kKT * DH;                 // [kQV][kKT+1]

  const int split = blockIdx.x, qg = blockIdx.y;
  const int r = blockIdx.z / Hkv, kh = blockIdx.z % Hkv;
  const int g = Hq / Hkv;
  if (r >= R) return;
  const int n0 = row_offset[r], nr = row_offset[r + 1] - n0;
  const int p0 = prefix_offset[r], P = prefix_offset[r + 1] - p0;
  if (n0 < 0 || nr < 1 || n0 + nr > N || p0 < 0 || P < 0 || p0 + P > total_prefix) {
    if (threadIdx.x == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  const int nvec = nr * g;
  const int vbase = qg * kQV;
  if (vbase >= nvec) return;
  const int k_begin = split * chunk;
  const int k_end = min(P, k_begin + chunk);

  const int tid = threadIdx.x;
  const int vec = tid >> 4, sub = tid & 15;
  const float scale = 1.4426950408889634f * rsqrtf(float(DH));  // base-2 scores
  for (int i = tid; i < kQV * DH; i += kThreads) {
    const int vv = i / DH, dd = i % DH, gv = vbase + vv;
    float x = 0.f;
    if (gv < nvec) {
      const int n = n0 + gv / g, h = kh * g + gv % g;
      x = to_f32(q[(size_t(n) * Hq + h) * DH + dd]) * scale;
    }
    Qs[vv * (DH + 1) + dd] = x;
  }

  constexpr int PER = DH / 16;
  float acc[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) acc[i] = 0.f;
  float m = -INFINITY, l = 0.f;

  for (int kb = k_begin; kb < k_end; kb += kKT) {
    const int nk = min(kKT, k_end - kb);
    __syncthreads();
    for (int i = tid; i < kKT * DH; i += kThreads) {
      const int j = i / DH, dd = i % DH;
      float kx = 0.f, vx = 0.f;
      if (j < nk) {
        const size_t idx = (size_t(p0 + kb + j) * Hkv + kh) * DH + dd;
        kx = to_f32(k_pre[idx]);
        vx = to_f32(v_pre[idx]);
      }
      Ks[j * (DH + 1) + dd] = kx;
      Vs[j * DH + dd] = vx;
    }
    __syncthreads();

    const float* qv = Qs + vec * (DH + 1);
    const float* k0 = Ks + sub * (DH + 1);
    const float* k1 = Ks + (sub + 16) * (DH + 1);
    float s0 = 0.f, s1 = 0.f;
#pragma unroll 8
    for (int dd = 0; dd < DH; ++dd) {
      const float x = qv[dd];
      s0 = fmaf(x, k0[dd], s0);
      s1 = fmaf(x, k1[dd], s1);
    }
    if (sub >= nk) s0 = -INFINITY;
    if (sub + 16 >= nk) s1 = -INFINITY;
    float tmax = fmaxf(s0, s1);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
    const float mn = fmaxf(m, tmax);            // finite: key 0 of the tile is valid
    const float corr = exp2f(m - mn);           // 0 on the first tile
    const float e0 = exp2f(s0 - mn), e1 = exp2f(s1 - mn);
    float psum = e0 + e1;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
    l = l * corr + psum;
    m = mn;
    Ps[vec * (kKT + 1) + sub] = e0;
    Ps[vec * (kKT + 1) + sub + 16] = e1;
    __syncwarp();
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] *= corr;
    for (int j = 0; j < nk; ++j) {
      const float pj = Ps[vec * (kKT + 1) + j];
      const float* vr = Vs + j * DH + sub;
#pragma unroll
      for (int i = 0; i < PER; ++i) acc[i] = fmaf(pj, vr[16 * i], acc[i]);
    }
  }

  const int gv = vbase + vec;
  if (gv < nvec) {
    const int n = n0 + gv / g, h = kh * g + gv % g;
    const size_t base = (size_t(split) * N + n) * Hq + h;
#pragma unroll
    for (int i = 0; i < PER; ++i) o_part[base * DH + sub + 16 * i] = acc[i];
    if (sub == 0) ml_part[base] = make_float2(m, l);
  }
}

// One warp per (row, query head): combine the prefix chunks, then the row's
// own causal candidate keys, and normalise.
template <typename T, int DH>
__global__ void __launch_bounds__(256)
attend_merge_kernel(const int32_t* __restrict__ row_req, const int32_t* __restrict__ row_cand,
                    const int32_t* __restrict__ cand_row_offset, int N, int R, int C, int Hq, int Hkv,
                    int splits, const T* __restrict__ q, const T* __restrict__ k_cand,
                    const T* __restrict__ v_cand, const float* __restrict__ o_part,
                    const float2* __restrict__ ml_part, T* __restrict__ o, int* status) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const long long idx = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (idx >= (long long)N * Hq) return;
  const int n = int(idx / Hq), h = int(idx % Hq);
  const int kh = h / (Hq / Hkv);
  constexpr int PER = DH / 32;
  float acc[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) acc[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int s = 0; s < splits; ++s) {
    const size_t base = (size_t(s) * N + n) * Hq + h;
    const float2 ml = ml_part[base];
    if (!(ml.y > 0.f)) continue;  // empty chunk
    const float mn = fmaxf(m, ml.x);
    const float a = exp2f(m - mn), b = exp2f(ml.x - mn);
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = acc[i] * a + o_part[base * DH + lane + 32 * i] * b;
    l = l * a + ml.y * b;
    m = mn;
  }
  const int c = row_cand[n];
  if (c >= 0) {
    const int r = row_req[n];
    const int first = (c < C) ? cand_row_offset[c] : -1;
    if (first < 0 || first > n || r < 0 || first - r - 1 < 0 || n - r - 1 >= N - R) {
      if (lane == 0) flag(status, JET_ERR_DEVICE);
    } else {
      const float scale = 1.4426950408889634f * rsqrtf(float(DH));  // base 2
      float qv[PER];
#pragma unroll
      for (int i = 0; i < PER; ++i) qv[i] = to_f32(q[(size_t(n) * Hq + h) * DH + lane + 32 * i]) * scale;
      for (int nn = first; nn <= n; ++nn) {
        const size_t kb = (size_t(nn - r - 1) * Hkv + kh) * DH + lane;
        float sp = 0.f;
#pragma unroll
        for (int i = 0; i < PER; ++i) sp = fmaf(qv[i], to_f32(k_cand[kb + 32 * i]), sp);
        const float sc = warp_sum(sp);
        const float mn = fmaxf(m, sc);
        const float a = exp2f(m - mn), b = exp2f(sc - mn);
#pragma unroll
        for (int i = 0; i < PER; ++i) acc[i] = acc[i] * a + b * to_f32(v_cand[kb + 32 * i]);
        l = l * a + b;
        m = mn;
      }
    }
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
  for (int i = 0; i < PER; ++i) o[(size_t(n) * Hq + h) * DH + lane + 32 * i] = from_f32<T>(acc[i] * inv);
}

template <typename T, int DH>
cudaError_t launch_typed(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                         const void* q, const void* k_pre, const void* v_pre, const void* k_cand,
                         const void* v_cand, void* o, void* ws, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  float* o_part = static_cast<float*>(ws);
  float2* ml_part = reinterpret_cast<float2*>(o_part + size_t(plan.splits) * n.N * d.Hq * DH);
  cudaError_t e;
  if (d.dtype == JET_DTYPE_BF16) {
    // the tensor-core path covers the candidates' own keys and the combine
    return launch_attend_tc(lay, d, plan, q, k_pre, v_pre, k_cand, v_cand, o, o_part, ml_part,
                            status, st);
  } else {
    const size_t smem = prefix_smem_bytes<DH>();
    e = cudaFuncSetAttribute(attend_prefix_kernel<T, DH>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return e;
    dim3 grid(plan.splits, plan.qgroups, unsigned(n.R * d.Hkv));
    e = launch_pdl(attend_prefix_kernel<T, DH>, grid, dim3(kThreads), smem, st, lay.prefix_offset,
                   lay.row_offset, n.R, n.N, n.total_prefix, d.Hq, d.Hkv, plan.chunk,
                   static_cast<const T*>(q), static_cast<const T*>(k_pre),
                   static_cast<const T*>(v_pre), o_part, ml_part, status);
  }
  if (e != cudaSuccess) return e;
  const long long warps = (long long)n.N * d.Hq;
  return launch_pdl(attend_merge_kernel<T, DH>, dim3(unsigned((warps + 7) / 8)), dim3(256), 0, st,
                    lay.row_req, lay.row_cand, lay.cand_row_offset, n.N, n.R, n.C, d.Hq, d.Hkv,
                    plan.splits, static_cast<const T*>(q), static_cast<const T*>(k_cand),
                    static_cast<const T*>(v_cand), o_part, ml_part, static_cast<T*>(o), status);
}

}  // namespace

AttnPlan attn_plan(const jet_sizes& n, const jet_dims& d) {
  AttnPlan p{};
  if (n.R <= 0 || n.N <= 0 || d.Hkv <= 0 || d.Hq <= 0) return p;
  const int g = d.Hq / d.Hkv;
  const bool tc = d.dtype == JET_DTYPE_BF16;
  const int gran = tc ? 64 : kKT;                 // keys per tile
  // query vectors per CTA: the tensor-core kernel takes whole rows (128 / g
  // rows of g heads), the float32 kernel kQV vectors
  const int qv = tc ? std::max(1, attn_tc_block() / g) * g : kQV;
  p.qgroups = (n.max_rows * g + qv - 1) / qv;
  // query blocks of an average request: blocks past a request's vectors exit
  // at once, so they do not count as work
  const long long avg_vecs = ((long long)n.N * g + n.R - 1) / n.R;
  const long long groups = (long long)n.R * d.Hkv * std::max<long long>(1, (avg_vecs + qv - 1) / qv);
  const int max_splits = std::max(1, (n.max_prefix + 63) / 64);
  int chunk;
  if (tc) {
    // the persistent kernel (one CTA per SM, longest items first) splits a
    // request's prefix into near-equal chunks: no shorter than kMinChunkTc keys
    // (an item's fixed cost - query block in, f32 partial out and read back by
    // the combine - is worth about five 64-key tiles), and no finer than half
    // of one SM's share of all key tiles, so that the schedule can balance
    const double avg_tiles = double(n.total_prefix) / n.R / 64.0 + 0.5;
    const double share = double(groups) * avg_tiles / kPlanSMs;  // tiles per SM
    chunk = std::max(kMinChunkTc, int(share / 2.0 + 0.999) * 64);
    chunk = std::min(chunk, max_splits * 64);  // one chunk holds the longest prefix
  } else {
    // about four CTAs per SM
    long long want = (kTargetCtas + groups - 1) / groups;
    int splits = int(std::min<long long>(std::max<long long>(want, 1), max_splits));
    chunk = (n.max_prefix + splits - 1) / splits;
    chunk = (chunk + gran - 1) / gran * gran;
  }
  p.chunk = chunk;
  p.splits = (n.max_prefix + chunk - 1) / chunk;
  const size_t vecs = size_t(p.splits) * n.N * d.Hq;
  p.bytes = vecs * d.d * sizeof(float) + vecs * sizeof(float2);
  // tensor-core path: a work list of (request, kv head, query block, chunk)
  // items plus two counters, 16-byte aligned, after the partials
  if (tc) p.bytes += 32 + 16 * size_t(n.R) * d.Hkv * p.qgroups * p.splits;
  return p;
}

cudaError_t launch_prefix_attend(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                                 const void* q, const void* k_pre, const void* v_pre,
                                 const void* k_cand, const void* v_cand, void* o, void* ws,
                                 int* status, cudaStream_t st) {
#define JET_ATT(T, DH) \
  return launch_typed<T, DH>(lay, d, plan, q, k_pre, v_pre, k_cand, v_cand, o, ws, status, st)
  if (d.dtype == JET_DTYPE_F32) {
    if (d.d == 64) JET_ATT(float, 64);
    if (d.d == 128) JET_ATT(float, 128);
    if (d.d == 256) JET_ATT(float, 256);
  } else {
    if (d.d == 64) JET_ATT(__nv_bfloat16, 64);
    if (d.d == 128) JET_ATT(__nv_bfloat16, 128);
    if (d.d == 256) JET_ATT(__nv_bfloat16, 256);
  }
#undef JET_ATT
  return cudaErrorInvalidValue;
}

}  // namespace jet
