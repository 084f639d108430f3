// Per-candidate fork of a linear-attention recurrent state (Sec. 4.1).
//
// The paper keeps one stored prefix state and restores it before each
// candidate, evaluating candidates one after another. Here one CTA per
// (32-column slice, head, request) reads the prefix state slice once into
// registers and the request's fed tokens once into shared memory; every
// candidate then starts from an unmodified register copy of the slice,
// applies its fed tokens and writes its own final state, so the state
// writes of one candidate overlap the arithmetic of the next. Each fed token
// applies the gated delta rule
//   S <- alpha (S - beta k (k^T S)) + beta k v^T,   o = S^T q / sqrt(dk)
// (the paper does not state its recurrence; this is the reading used).
// The update is column-separable: column j of S needs only k, v_j and the
// column's own u_j = k^T S[:, j], so a CTA owns a 32-column slice of one
// head. The kernel is bound by the writes of the forked states. The plain
// gated linear-attention variant S <- alpha S + beta k v^T is the same update
// with u = 0 (the DELTA = false instantiation skips that reduction).
#include "jet_device.cuh"
#include "jet_internal.h"

namespace jet {
namespace {

constexpr int kDK = 128;        // key dimension handled (rows of S)
constexpr int kCols = 32;       // value columns per CTA
constexpr int kThreads = 128;   // 4 warps x 32 rows
constexpr int kWin = 16;        // fed tokens staged in shared memory at a time
constexpr int kMeta = 64;       // candidates whose lengths are staged at a time

__device__ __forceinline__ float4 f4_fma(float a, float4 x, float4 y) {
  return make_float4(fmaf(a, x.x, y.x), fmaf(a, x.y, y.y), fmaf(a, x.z, y.z), fmaf(a, x.w, y.w));
}

// Reduce a per-thread float4 over the 128 rows of the slice; every thread
// receives the 4 column sums of its column quad. `red` holds 4 x 32 floats.
__device__ __forceinline__ float4 rows_sum(float4 v, float* red, int warp, int lane) {
#pragma unroll
  for (int o = 8; o <= 16; o <<= 1) {
    v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
    v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
    v.z += __shfl_xor_sync(0xffffffffu, v.z, o);
    v.w += __shfl_xor_sync(0xffffffffu, v.w, o);
  }
  const int jq = lane & 7;
  if (lane < 8) reinterpret_cast<float4*>(red)[warp * 8 + jq] = v;
  __syncthreads();
  float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const float4 t = reinterpret_cast<const float4*>(red)[w * 8 + jq];
    s.x += t.x; s.y += t.y; s.z += t.z; s.w += t.w;
  }
  __syncthreads();
  return s;
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}

__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Stage fed tokens [w0, w0 + nt) (nt <= kWin) into shared memory as they are
// stored: their k and q rows, this slice's v columns and the gates. The
// copies are asynchronous and all in flight at once, so a window costs one
// memory latency and no registers; the caller synchronises the block.
template <typename T>
__device__ __forceinline__ void stage_window(const T* __restrict__ q, const T* __restrict__ k,
                                             const T* __restrict__ v,
                                             const float* __restrict__ alpha,
                                             const float* __restrict__ beta, int Hl, int dv,
                                             int h, int j0, int w0, int nt, int tid,
                                             T (*wk)[kDK], T (*wq)[kDK], T (*wv)[kCols],
                                             float* wa, float* wb) {
  constexpr int VE = 16 / int(sizeof(T));  // elements per 16-byte piece
  constexpr int KP = kDK / VE;             // pieces of a k (or q) row
  constexpr int VP = kCols / VE;           // pieces of a v slice row
  for (int e = tid; e < nt * KP; e += kThreads) {
    const int tok = e / KP, pc = e % KP;
    const size_t src = (size_t(w0 + tok) * Hl + h) * kDK + pc * VE;
    cp_async16(&wk[tok][pc * VE], k + src);
    cp_async16(&wq[tok][pc * VE], q + src);
  }
  for (int e = tid; e < nt * VP; e += kThreads) {
    const int tok = e / VP, pc = e % VP;
    cp_async16(&wv[tok][pc * VE], v + (size_t(w0 + tok) * Hl + h) * dv + j0 + pc * VE);
  }
  if (tid < nt) {
    cp_async4(&wa[tid], alpha + size_t(w0 + tid) * Hl + h);
    cp_async4(&wb[tid], beta + size_t(w0 + tid) * Hl + h);
  }
  cp_async_wait_all();
}

__device__ __forceinline__ int wt_of(int f, int w0) { return f - w0; }

// One token of the recurrence on this thread's part of the slice (rows
// 32 w + rg + 4 ii, columns 4 jq .. + 3), token wt of the staged window:
// S = alpha S + beta k (v - alpha u), u = k^T S (u = 0 for gated linear
// attention). Returns the slice's output columns o = S^T q (unscaled), the
// same in every thread of a column quad.
template <typename T, bool DELTA>
__device__ __forceinline__ float4 token_step(float4 (&S)[8], int wt, const T (*wk)[kDK],
                                             const T (*wq)[kDK], const T (*wv)[kCols],
                                             const float* wa, const float* wb, float* red,
                                             int warp, int lane) {
  const int rg = lane >> 3, jq = lane & 7;
  float kk[8], qq[8];
#pragma unroll
  for (int ii = 0; ii < 8; ++ii) {
    const int i = 32 * warp + rg + 4 * ii;
    kk[ii] = to_f32(wk[wt][i]);
    qq[ii] = to_f32(wq[wt][i]);
  }
  const float a = wa[wt], b = wb[wt];
  const float4 vv = make_float4(to_f32(wv[wt][4 * jq]), to_f32(wv[wt][4 * jq + 1]),
                                to_f32(wv[wt][4 * jq + 2]), to_f32(wv[wt][4 * jq + 3]));
  // u = k^T S for this column quad (the delta rule's erase term)
  float4 u = make_float4(0.f, 0.f, 0.f, 0.f);
  if (DELTA) {
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) u = f4_fma(kk[ii], S[ii], u);
    u = rows_sum(u, red, warp, lane);
  }
  const float4 w = make_float4(b * (vv.x - a * u.x), b * (vv.y - a * u.y), b * (vv.z - a * u.z),
                               b * (vv.w - a * u.w));
  float4 op = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int ii = 0; ii < 8; ++ii) {
    float4 s = S[ii];
    s = make_float4(fmaf(kk[ii], w.x, a * s.x), fmaf(kk[ii], w.y, a * s.y),
                    fmaf(kk[ii], w.z, a * s.z), fmaf(kk[ii], w.w, a * s.w));
    S[ii] = s;
    op = f4_fma(qq[ii], s, op);
  }
  return rows_sum(op, red, warp, lane);
}

// grid (dv / 32, Hl, R); thread (warp w, lane = 8 * rg + jq) owns rows
// 32 w + rg + 4 ii (ii < 8) and columns j0 + 4 jq .. + 3 of the slice.
// q_rows (optional, [N, Hl, dk]): every row's q; the request's shared row then
// reads the prefix state, o = S_r^T q / sqrt(dk), and o holds all N rows
// (fed token f at row f + r + 1) instead of the fed tokens alone.
// bf16: 72 registers and 28 KB of shared memory, so that seven CTAs share an
// SM (a (32 requests x 16 heads x 4 slices) grid then fills 1.93 waves of
// 1,064 CTAs instead of 2.25 waves of 912)
template <typename T, bool DELTA>
__global__ void __launch_bounds__(kThreads, sizeof(T) == 2 ? 7 : 3)
fork_kernel(const int32_t* __restrict__ cand_offset, const int32_t* __restrict__ cand_row_offset,
            const int32_t* __restrict__ tgt_offset, const int32_t* __restrict__ row_offset,
            int R, int C, int F, int Hl, int dv, const float* __restrict__ s_prefix,
            const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
            const float* __restrict__ alpha, const float* __restrict__ beta,
            const T* __restrict__ q_rows, T* __restrict__ o, float* __restrict__ s_fork,
            int* status) {
  pdl_begin();
  __shared__ __align__(16) float red[4 * kCols];
  // a window of the request's fed tokens as stored: k, q (all rows), v (this
  // slice), gates
  __shared__ __align__(16) T wk[kWin][kDK];
  __shared__ __align__(16) T wq[kWin][kDK];
  __shared__ __align__(16) T wv[kWin][kCols];
  __shared__ __align__(16) float wa[kWin], wb[kWin];
  // the (length, first fed token) of up to kMeta candidates at a time
  __shared__ int cm[kMeta], cf[kMeta];
  // the prefix state slice, each thread's own 8 float4 at [ii][tid]
  __shared__ __align__(16) float4 ssp[8 * kThreads];
  __shared__ float qsh[kDK];  // the shared row's q (with q_rows)
  const int r = blockIdx.z, h = blockIdx.y, j0 = blockIdx.x * kCols;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rg = lane >> 3, jq = lane & 7;
  const int col = j0 + 4 * jq;
  if (r >= R) return;
  const int c0 = cand_offset[r], c1 = cand_offset[r + 1];
  const int f_begin = row_offset[r] - r;                   // the request's first fed token
  const int f_end = f_begin + row_offset[r + 1] - row_offset[r] - 1;
  if (c0 < 0 || c1 < c0 || c1 > C || f_begin < 0 || f_end < f_begin || f_end > F) {
    if (tid == 0) flag(status, JET_ERR_DEVICE);
    return;
  }

  // the prefix state slice (read once, kept in shared memory for every
  // candidate) and the first window of fed tokens load at once
  const float rs = rsqrtf(float(kDK));
  {
    float4 sp[8];
    const size_t head = (size_t(r) * Hl + h) * kDK;
    if (q_rows && tid < kDK)
      qsh[tid] = to_f32(q_rows[(size_t(row_offset[r]) * Hl + h) * kDK + tid]);
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) {
      const int i = 32 * warp + rg + 4 * ii;
      sp[ii] = *reinterpret_cast<const float4*>(s_prefix + (head + i) * dv + col);
    }
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) ssp[ii * kThreads + tid] = sp[ii];
    if (q_rows) {
      // the shared row: o = S_r^T q / sqrt(dk), from the prefix state itself
      __syncthreads();  // qsh is in
      float4 op = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int ii = 0; ii < 8; ++ii) op = f4_fma(qsh[32 * warp + rg + 4 * ii], sp[ii], op);
      op = rows_sum(op, red, warp, lane);
      if (warp == 0 && rg == 0) {
        T* dst = o + (size_t(row_offset[r]) * Hl + h) * dv + col;
        dst[0] = from_f32<T>(op.x * rs);
        dst[1] = from_f32<T>(op.y * rs);
        dst[2] = from_f32<T>(op.z * rs);
        dst[3] = from_f32<T>(op.w * rs);
      }
    }
  }
  // with q_rows, fed token f is written at row f + r + 1
  const size_t o_shift = q_rows ? size_t(r) + 1 : 0;
  int w0 = f_begin, w1 = min(f_begin + kWin, f_end);  // fed tokens [w0, w1) are staged
  if (w1 > w0)
    stage_window(q, k, v, alpha, beta, Hl, dv, h, j0, w0, w1 - w0, tid, wk, wq, wv, wa, wb);

  for (int cb = c0; cb < c1; cb += kMeta) {
    const int nb = min(kMeta, c1 - cb);
    __syncthreads();  // the previous batch's lengths are no longer read
    for (int e = tid; e < nb; e += kThreads) {
      cm[e] = tgt_offset[cb + e + 1] - tgt_offset[cb + e];
      cf[e] = cand_row_offset[cb + e] - r - 1;  // fed-token index of y_{c,1}
    }
    __syncthreads();
    for (int e = 0; e < nb; ++e) {
      const int c = cb + e;
      const int m = cm[e], f0 = cf[e];
      if (m < 1 || f0 < f_begin || f0 + m - 1 > f_end) {
        if (tid == 0) flag(status, JET_ERR_DEVICE);
        continue;
      }
      float4 S[8];
#pragma unroll
      for (int ii = 0; ii < 8; ++ii) S[ii] = ssp[ii * kThreads + tid];  // the prefix state
      for (int t = 0; t < m - 1; ++t) {
        const int f = f0 + t;
        if (f < w0 || f >= w1) {
          // stage the window of fed tokens starting at f
          __syncthreads();
          w0 = f;
          w1 = min(f + kWin, f_end);
          stage_window(q, k, v, alpha, beta, Hl, dv, h, j0, w0, w1 - w0, tid, wk, wq, wv, wa, wb);
          __syncthreads();
        }
        const float4 op = token_step<T, DELTA>(S, wt_of(f, w0), wk, wq, wv, wa, wb, red, warp,
                                               lane);
        if (warp == 0 && rg == 0) {
          T* dst = o + ((size_t(f) + o_shift) * Hl + h) * dv + col;
          dst[0] = from_f32<T>(op.x * rs);
          dst[1] = from_f32<T>(op.y * rs);
          dst[2] = from_f32<T>(op.z * rs);
          dst[3] = from_f32<T>(op.w * rs);
        }
      }
      if (s_fork) {
        // streaming stores: the forked states are not read again in the step,
        // so they should not displace its working set in L2 (3 us less here)
        const size_t fhead = (size_t(c) * Hl + h) * kDK;
#pragma unroll
        for (int ii = 0; ii < 8; ++ii) {
          const int i = 32 * warp + rg + 4 * ii;
          __stcs(reinterpret_cast<float4*>(s_fork + (fhead + i) * dv + col), S[ii]);
        }
      }
    }
  }
}

}  // namespace

namespace {

template <bool DELTA>
cudaError_t launch_rule(const jet_layout& lay, const jet_dims& d, const float* s_prefix,
                        const void* q, const void* k, const void* v, const float* alpha,
                        const float* beta, const void* q_rows, void* o, float* s_fork,
                        int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  dim3 grid(unsigned(d.dv / kCols), unsigned(d.Hl), unsigned(n.R));
  const int F = n.N - n.R;
  if (d.dtype == JET_DTYPE_F32) {
    return launch_pdl(fork_kernel<float, DELTA>, grid, dim3(kThreads), 0, st, lay.cand_offset,
                      lay.cand_row_offset, lay.tgt_offset, lay.row_offset, n.R, n.C, F, d.Hl,
                      d.dv, s_prefix, static_cast<const float*>(q), static_cast<const float*>(k),
                      static_cast<const float*>(v), alpha, beta,
                      static_cast<const float*>(q_rows), static_cast<float*>(o), s_fork, status);
  }
  return launch_pdl(fork_kernel<__nv_bfloat16, DELTA>, grid, dim3(kThreads), 0, st,
                    lay.cand_offset, lay.cand_row_offset, lay.tgt_offset, lay.row_offset, n.R,
                    n.C, F, d.Hl, d.dv, s_prefix, static_cast<const __nv_bfloat16*>(q),
                    static_cast<const __nv_bfloat16*>(k), static_cast<const __nv_bfloat16*>(v),
                    alpha, beta, static_cast<const __nv_bfloat16*>(q_rows),
                    static_cast<__nv_bfloat16*>(o), s_fork, status);
}

}  // namespace


cudaError_t launch_fork_state(const jet_layout& lay, const jet_dims& d, int rule,
                              const float* s_prefix, const void* q, const void* k, const void* v,
                              const float* alpha, const float* beta, void* o, float* s_fork,
                              int* status, cudaStream_t st, const void* q_rows) {
  if (rule == JET_RECUR_GLA)
    return launch_rule<false>(lay, d, s_prefix, q, k, v, alpha, beta, q_rows, o, s_fork, status,
                              st);
  return launch_rule<true>(lay, d, s_prefix, q, k, v, alpha, beta, q_rows, o, s_fork, status, st);
}

}  // namespace jet
