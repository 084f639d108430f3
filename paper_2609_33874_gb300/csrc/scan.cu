// Prefill of a linear-attention layer's recurrent state: every request's
// prefix tokens fed in order through the recurrence (the gated delta rule,
// or plain gated linear attention), producing each token's output and the
// state s_prefix that the candidates fork from (Sec. 4.1). The machinery it
// shares with the fork is in recur.cuh.
//
// The scan is sequential in the tokens of a request, so the parallelism is
// (request, head, value column). Column j of S needs only k, v_j and its own
// u_j = k^T S[:, j], so one CTA owns 64 columns of one head of one request
// and keeps that 128 x 64 slice of S in registers for the whole prefix:
// thread (warp w, lane = 8 p + c) holds rows 32 p .. 32 p + 31 and columns
// 16 w + 2 c, + 1. One sweep over the thread's rows per token applies the
// update of token t and accumulates both o_t = S_t^T q_t and the next
// token's u_{t+1} = S_t^T k_{t+1}, so each state element costs three FMAs a
// token and the two row sums reduce together over the 4 lanes of a column
// pair with shuffles (no block barrier inside the token loop). The decay is
// carried as one scalar gain G with S = G S~ (folded back into S~ before it
// underflows), so it costs no multiply per element. Tokens are staged 16 at a
// time: asynchronous copies of the next window land in a raw buffer while the
// current window's tokens run, and are widened to fp32 (exact for bf16) at
// the window boundary.
#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

#include "recur.cuh"

// grid (ceil(dv / 64), Hl, R). S starts from s_init (zeros when null); the
// outputs o[p] = S_p^T q_p / sqrt(dk) of every prefix token and the final
// state are written.
template <typename T, bool DELTA>
__global__ void __launch_bounds__(kThreads, sizeof(T) == 2 ? 4 : 3)
scan_kernel(const int32_t* __restrict__ prefix_offset, int R, int total, int Hl, int dv,
            const float* __restrict__ s_init, const T* __restrict__ q, const T* __restrict__ k,
            const T* __restrict__ v, const float* __restrict__ alpha,
            const float* __restrict__ beta, T* __restrict__ o, float* __restrict__ s_out,
            int* status) {
  pdl_begin();
  __shared__ __align__(16) float fk[kWin + 1][kPad];
  __shared__ __align__(16) float fq[kWin][kPad];
  __shared__ __align__(16) float fv[kWin][kCols];
  __shared__ float fa[kWin], fb[kWin];
  __shared__ __align__(16) RawWindow<T> raw;
  const int r = blockIdx.z, h = blockIdx.y, j0 = blockIdx.x * kCols;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // lanes of a row group are adjacent, so a staged k or q read is one
  // address per quarter-warp
  const int p = lane >> 3, c = lane & 7;
  const int cw = 16 * warp + 2 * c;  // this thread's first column within the CTA
  const bool active = j0 + 16 * warp < dv;  // dv % 64 == 32: the last CTA's upper warps idle
  if (r >= R) return;
  const int p0 = prefix_offset[r], p1 = prefix_offset[r + 1];
  if (p0 < 0 || p1 < p0 || p1 > total) {
    if (tid == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  const size_t head = (size_t(r) * Hl + h) * kDK;
  float2 s[kRows];
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    const size_t at = (head + kRows * p + i) * dv + j0 + cw;
    s[i] = (s_init && active) ? *reinterpret_cast<const float2*>(s_init + at)
                              : make_float2(0.f, 0.f);
  }
  float G = 1.f;  // S = G * s
  const float rs = rsqrtf(float(kDK));
  const int rb = padded(kRows * p);  // this thread's rows in a staged k or q row
  const bool writer = (lane & 16) == 0;
  T* out = o + size_t(p0) * Hl * dv + size_t(h) * dv + j0 + cw + ((lane >> 3) & 1);
  const size_t out_step = size_t(Hl) * dv;

  raw.fetch(q, k, v, alpha, beta, Hl, dv, h, j0, p0, min(kWin, p1 - p0), min(kWin + 1, p1 - p0),
            tid);
  float2 u = make_float2(0.f, 0.f);  // k^T S of the next token (delta rule)
  for (int w0 = p0; w0 < p1; w0 += kWin) {
    const int nt = min(kWin, p1 - w0);
    cp_async_wait_all();
    __syncthreads();  // the window has landed; the previous one is no longer read
    raw.widen(fk, fq, fv, fa, fb, min(kWin + 1, p1 - w0), tid);
    __syncthreads();  // widened; the raw buffer is free again
    if (w0 + kWin < p1)
      raw.fetch(q, k, v, alpha, beta, Hl, dv, h, j0, w0 + kWin, min(kWin, p1 - w0 - kWin),
                min(kWin + 1, p1 - w0 - kWin), tid);
    if (!active) continue;
    // u of the prefix's first token, from the initial state
    if (DELTA && w0 == p0) u = k_dot_s(s, &fk[0][rb], G);
    for (int t = 0; t < nt; ++t) {
      const float2 vv = *reinterpret_cast<const float2*>(&fv[t][cw]);
      // the next token's k is the staged row t + 1 (zero past the prefix)
      const float z = recur_token<DELTA, true>(s, G, u, fa[t], fb[t], vv, &fk[t][rb], &fq[t][rb],
                                               &fk[t + 1][rb], lane);
      if (writer) out[size_t(t) * out_step] = from_f32<T>(z * rs);
    }
    out += size_t(kWin) * out_step;
  }
  if (!active) return;
#pragma unroll
  for (int i = 0; i < kRows; ++i) {
    *reinterpret_cast<float2*>(s_out + (head + kRows * p + i) * dv + j0 + cw) =
        make_float2(G * s[i].x, G * s[i].y);
  }
}

}  // namespace

cudaError_t launch_prefill_state(const jet_layout& lay, const jet_dims& d, int rule,
                                 const float* s_init, const void* q, const void* k, const void* v,
                                 const float* alpha, const float* beta, void* o, float* s_out,
                                 int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  // bf16 with 128 x 128 states: the chunked form on the tensor cores
  if (scan_tc_supported(d))
    return launch_scan_tc(lay, d, rule, s_init, q, k, v, alpha, beta, o, s_out, status, st);
  dim3 grid(unsigned((d.dv + kCols - 1) / kCols), unsigned(d.Hl), unsigned(n.R));
#define JET_SCAN(T, DELTA)                                                                   \
  return launch_pdl(scan_kernel<T, DELTA>, grid, dim3(kThreads), 0, st, lay.prefix_offset, n.R, \
                    n.total_prefix, d.Hl, d.dv, s_init, static_cast<const T*>(q),             \
                    static_cast<const T*>(k), static_cast<const T*>(v), alpha, beta,          \
                    static_cast<T*>(o), s_out, status)
  const bool delta = rule != JET_RECUR_GLA;
  if (d.dtype == JET_DTYPE_F32) {
    if (delta) JET_SCAN(float, true);
    JET_SCAN(float, false);
  }
  if (delta) JET_SCAN(__nv_bfloat16, true);
  JET_SCAN(__nv_bfloat16, false);
#undef JET_SCAN
}

}  // namespace jet
