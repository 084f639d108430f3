// Log-sum-exp merge, token log-probabilities, candidate scores and the
// decision rules.
//
//   lse_n   = ln 2 (m + log2 sum_tiles s_i 2^(m_i - m)) over the base-2 per-tile
//             partials (Eq. 2: a = max_v z, lse = a + log sum_v exp(z_v - a))
//   l_{c,t} = z_{c,t,y} - lse of its row                      (Eq. 1, Eq. 2)
//   s(c|x)  = sum_t l_{c,t}, summed in t order                (Eq. 3)
//   q(c)    = exp(s_c - M) / sum_d exp(s_d - M), M = max s     (Eq. 4)
//   choice  = argmax_c s_c, ties to the lowest index          (Eq. 5, Sec. 3.3)
//   nll     = -log sum_{c: gold label text} q(c)               (Sec. 3.3, Sec. 5.1)
//   correct = the chosen label carries the gold answer text    (Sec. 5.1)
#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

// one block per row (blockDim.x a multiple of 32, at most kLseThreads);
// coalesced reads of the row's partials part[n][0..vtiles). 512 threads: a
// row's ~1,200 partials are then two or three loads a thread, all in flight
// at once (with 128 threads the merge was latency-bound: 1.5-2 us more a step)
constexpr int kLseThreads = 512;
__global__ void __launch_bounds__(kLseThreads)
lse_kernel(const float2* __restrict__ part, int vtiles, int N, float* __restrict__ lse) {
  pdl_begin();
  __shared__ float2 red[kLseThreads / 32];
  const int n = blockIdx.x;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float2* p = part + size_t(n) * vtiles;
  float m = -INFINITY, s = 0.f;
#pragma unroll 4
  for (int vt = threadIdx.x; vt < vtiles; vt += blockDim.x) {
    const float2 x = p[vt];
    ms_combine2(m, s, x.x, x.y);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    ms_combine2(m, s, m2, s2);
  }
  if (lane == 0) red[warp] = make_float2(m, s);
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int i = 1; i < int(blockDim.x / 32); ++i) ms_combine2(m, s, red[i].x, red[i].y);
    lse[n] = (m + log2f(s)) * 0.6931471805599453f;  // partials are base 2
  }
}

// one warp per candidate: lane t reads target t's logit and its row's lse
// (32 targets at a time, all loads in flight together), then lane 0 adds the
// log-probabilities in t order
__global__ void __launch_bounds__(256)
finish_kernel(const int32_t* __restrict__ tgt_offset, const int32_t* __restrict__ tgt_row, int C,
              int N, int T_, const float* __restrict__ z_tgt, const float* __restrict__ lse,
              float* __restrict__ tok_logprob, float* __restrict__ cand_score, int* status) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (c >= C) return;
  const int j0 = tgt_offset[c], j1 = tgt_offset[c + 1];
  if (j0 < 0 || j1 < j0 || j1 > T_) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  float acc = 0.f;
  for (int jb = j0; jb < j1; jb += 32) {
    const int j = jb + lane;
    float ell = 0.f;
    if (j < j1) {
      const int n = tgt_row[j];
      if (n < 0 || n >= N) {
        flag(status, JET_ERR_DEVICE);
      } else {
        ell = z_tgt[j] - lse[n];
        tok_logprob[j] = ell;
      }
    }
    const int cnt = min(32, j1 - jb);
    for (int t = 0; t < cnt; ++t) acc += __shfl_sync(0xffffffffu, ell, t);
  }
  if (lane == 0) cand_score[c] = acc;
}

// one warp per request
__global__ void __launch_bounds__(256)
decide_kernel(const int32_t* __restrict__ cand_offset, int R, int C, int mode,
              const float* __restrict__ s, float* __restrict__ q, int32_t* __restrict__ choice,
              float* __restrict__ value, int* status) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= R) return;
  const int c0 = cand_offset[r], c1 = cand_offset[r + 1];
  if (c0 < 0 || c1 <= c0 || c1 > C) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  // M = max s, and the lowest index attaining it
  float best = -INFINITY;
  int arg = 0x7fffffff;
  for (int c = c0 + lane; c < c1; c += 32) {
    const float v = s[c];
    if (v > best) {  // strict: a lane keeps its lowest index among equals
      best = v;
      arg = c - c0;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oa = __shfl_xor_sync(0xffffffffu, arg, o);
    if (ob > best || (ob == best && oa < arg)) {
      best = ob;
      arg = oa;
    }
  }
  if (arg == 0x7fffffff) arg = 0;  // no finite score: fall back to the first candidate
  float sum = 0.f;
  for (int c = c0 + lane; c < c1; c += 32) sum += __expf(s[c] - best);
  sum = warp_sum(sum);
  const float inv = 1.f / sum;
  float ev = 0.f;
  for (int c = c0 + lane; c < c1; c += 32) {
    const float qc = __expf(s[c] - best) * inv;
    q[c] = qc;
    ev += float(c - c0) * qc;
  }
  ev = warp_sum(ev);
  if (lane == 0) {
    choice[r] = arg;
    if (mode == JET_DECIDE_BINARY)
      value[r] = (c1 - c0 == 2) ? __expf(s[c0 + 1] - best) * inv : __int_as_float(0x7fc00000);
    else if (mode == JET_DECIDE_ORDINAL)
      value[r] = ev;
    else
      value[r] = inv;  // q of the argmax: exp(0) / sum
  }
}

// one warp per request: nll = lse(all s) - lse(gold s), each log-sum-exp
// shifted by its own maximum, so a gold probability far below float32's
// range still gives a finite value
__global__ void __launch_bounds__(256)
evaluate_kernel(const int32_t* __restrict__ cand_offset, int R, int C,
                const float* __restrict__ s, const int32_t* __restrict__ choice,
                const uint8_t* __restrict__ gold, float* __restrict__ nll,
                int32_t* __restrict__ correct, int* status) {
  pdl_begin();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (r >= R) return;
  const int c0 = cand_offset[r], c1 = cand_offset[r + 1];
  if (c0 < 0 || c1 <= c0 || c1 > C) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  float M = -INFINITY, Mg = -INFINITY;
  for (int c = c0 + lane; c < c1; c += 32) {
    M = fmaxf(M, s[c]);
    if (gold[c]) Mg = fmaxf(Mg, s[c]);
  }
  M = warp_max(M);
  Mg = warp_max(Mg);
  float all = 0.f, in_gold = 0.f;
  for (int c = c0 + lane; c < c1; c += 32) {
    all += expf(s[c] - M);
    if (gold[c]) in_gold += expf(s[c] - Mg);
  }
  all = warp_sum(all);
  in_gold = warp_sum(in_gold);
  if (lane == 0) {
    // no gold candidate: Mg = -inf and the gold probability is zero
    // (M - Mg) first: exact for nearby maxima, it keeps the offset of the
    // scores out of the rounding of the small log terms
    nll[r] = Mg > -INFINITY ? (M - Mg) + (logf(all) - logf(in_gold)) : INFINITY;
    const int k = choice[r];
    if (k < 0 || k >= c1 - c0) {
      flag(status, JET_ERR_DEVICE);
      correct[r] = 0;
    } else {
      correct[r] = gold[c0 + k] ? 1 : 0;
    }
  }
}

}  // namespace

ScorePlan score_plan(const jet_sizes& n) {
  ScorePlan p{};
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  p.vtiles = (n.V + kVocabTile - 1) / kVocabTile;
  p.part_off = 0;
  p.ztgt_off = up(size_t(p.vtiles) * n.N * sizeof(float2));
  p.lse_off = p.ztgt_off + up(size_t(n.T) * sizeof(float));
  p.bytes = p.lse_off + up(size_t(n.N) * sizeof(float));
  return p;
}

cudaError_t launch_score_finish(const jet_layout& lay, const ScorePlan& plan, void* ws,
                                float* tok_logprob, float* cand_score, int* status,
                                cudaStream_t st) {
  const jet_sizes& n = lay.n;
  char* base = static_cast<char*>(ws);
  const float2* part = reinterpret_cast<const float2*>(base + plan.part_off);
  const float* z_tgt = reinterpret_cast<const float*>(base + plan.ztgt_off);
  float* lse = reinterpret_cast<float*>(base + plan.lse_off);
  cudaError_t e =
      launch_pdl(lse_kernel, dim3(unsigned(n.N)), dim3(kLseThreads), 0, st, part, plan.vtiles,
                 n.N, lse);
  if (e != cudaSuccess) return e;
  return launch_pdl(finish_kernel, dim3(unsigned((n.C + 7) / 8)), dim3(256), 0, st,
                    lay.tgt_offset, lay.tgt_row, n.C, n.N, n.T, z_tgt, lse, tok_logprob,
                    cand_score, status);
}

cudaError_t launch_evaluate(const jet_layout& lay, const float* cand_score, const int32_t* choice,
                            const uint8_t* gold, float* nll, int32_t* correct, int* status,
                            cudaStream_t st) {
  const jet_sizes& n = lay.n;
  return launch_pdl(evaluate_kernel, dim3(unsigned((n.R + 7) / 8)), dim3(256), 0, st,
                    lay.cand_offset, n.R, n.C, cand_score, choice, gold, nll, correct, status);
}

cudaError_t launch_decide(const jet_layout& lay, int mode, const float* cand_score, float* q,
                          int32_t* choice, float* value, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  return launch_pdl(decide_kernel, dim3(unsigned((n.R + 7) / 8)), dim3(256), 0, st,
                    lay.cand_offset, n.R, n.C, mode, cand_score, q, choice, value, status);
}

}  // namespace jet
