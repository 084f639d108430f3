// Prefill of a linear-attention layer's recurrent state: every request's
// prefix tokens fed in order through the recurrence (the gated delta rule,
// or plain gated linear attention), producing each token's output and the
// state s_prefix that the candidates fork from (Sec. 4.1).
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

constexpr int kDK = 128;                       // rows of S (key dimension)
constexpr int kCols = 64;                      // value columns per CTA
constexpr int kThreads = 128;                  // 4 warps x 16 columns
constexpr int kWin = 16;                       // prefix tokens staged at a time
constexpr int kRows = 32;                      // rows of S per thread
constexpr int kPad = kDK + (kDK / kRows) * 4;  // staged row: a 4-float gap per 32 rows
constexpr float kMinGain = 0x1p-32f;           // fold G into S~ below this
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ int padded(int i) { return i + (i / kRows) * 4; }

__device__ __forceinline__ float4 f4_fma(float a, float4 x, float4 y) {
  return make_float4(fmaf(a, x.x, y.x), fmaf(a, x.y, y.y), fmaf(a, x.z, y.z), fmaf(a, x.w, y.w));
}

// Both column sums of a column pair over its 4 lanes (lane bits 3, 4), in
// every lane (butterfly: the four lanes add in the same pairs, so they hold
// identical values).
__device__ __forceinline__ float2 pair_sum_all(float2 x) {
  x.x += __shfl_xor_sync(kFull, x.x, 8);
  x.y += __shfl_xor_sync(kFull, x.y, 8);
  x.x += __shfl_xor_sync(kFull, x.x, 16);
  x.y += __shfl_xor_sync(kFull, x.y, 16);
  return x;
}

// The column pair's sums over its 4 lanes, one column per lane: lane bit 3
// selects the column whose total the lane receives.
__device__ __forceinline__ float pair_sum_one(float2 x, int lane) {
  const bool e = (lane >> 3) & 1;
  float z = (e ? x.y : x.x) + __shfl_xor_sync(kFull, e ? x.x : x.y, 8);
  z += __shfl_xor_sync(kFull, z, 16);
  return z;
}

// One sweep over the thread's 32 rows for token t: S~ += k_t w^T, then
// o += q_t^T S~ and (NEXT) u += k_{t+1}^T S~ on the updated rows.
template <bool NEXT>
__device__ __forceinline__ void sweep(float2 (&s)[kRows], const float* kt, const float* qt,
                                      const float* kn, float2 w, float2& op, float2& un) {
  float2 o0 = make_float2(0.f, 0.f), o1 = o0, u0 = o0, u1 = o0;
#pragma unroll
  for (int m = 0; m < kRows / 4; ++m) {
    const float4 k4 = *reinterpret_cast<const float4*>(kt + 4 * m);
    const float4 q4 = *reinterpret_cast<const float4*>(qt + 4 * m);
    float4 n4 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (NEXT) n4 = *reinterpret_cast<const float4*>(kn + 4 * m);
    const float kr[4] = {k4.x, k4.y, k4.z, k4.w};
    const float qr[4] = {q4.x, q4.y, q4.z, q4.w};
    const float nr[4] = {n4.x, n4.y, n4.z, n4.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2& x = s[4 * m + i];
      x.x = fmaf(kr[i], w.x, x.x);
      x.y = fmaf(kr[i], w.y, x.y);
      float2& o = (i & 1) ? o1 : o0;
      o.x = fmaf(qr[i], x.x, o.x);
      o.y = fmaf(qr[i], x.y, o.y);
      if (NEXT) {
        float2& u = (i & 1) ? u1 : u0;
        u.x = fmaf(nr[i], x.x, u.x);
        u.y = fmaf(nr[i], x.y, u.y);
      }
    }
  }
  op = make_float2(o0.x + o1.x, o0.y + o1.y);
  if (NEXT) un = make_float2(u0.x + u1.x, u0.y + u1.y);
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

__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// A window of prefix tokens as stored (k and q rows, this CTA's v columns,
// the gates), filled by asynchronous copies while the previous window's
// tokens run, then widened into the fp32 buffers the token loop reads.
template <typename T>
struct RawWindow {
  static constexpr int VE = 16 / int(sizeof(T));              // elements per 16-byte piece
  static constexpr int KPR = kDK / VE;                        // pieces per k or q row
  static constexpr int NKQ = 2 * kWin * KPR / kThreads;       // k and q pieces per thread
  static constexpr int VPR = kCols / VE;                      // pieces per v row
  static constexpr int NV = kWin * VPR / kThreads;            // v pieces per thread
  static_assert(NKQ * kThreads == 2 * kWin * KPR && NV * kThreads == kWin * VPR, "split");
  T k[kWin + 1][kDK];  // one more k row: the next window's first token
  T q[kWin][kDK];
  T v[kWin][kCols];
  float g[2][kWin];  // alpha, beta

  // issue the copies of tokens [w0, w0 + nt), and of k for token w0 + kWin
  // when it exists (nk = kWin + 1)
  __device__ __forceinline__ void fetch(const T* __restrict__ qg, const T* __restrict__ kg,
                                        const T* __restrict__ vg, const float* __restrict__ alpha,
                                        const float* __restrict__ beta, int Hl, int dv, int h,
                                        int j0, int w0, int nt, int nk, int tid) {
    if (tid < KPR && kWin < nk)
      cp_async16(&k[kWin][tid * VE], kg + (size_t(w0 + kWin) * Hl + h) * kDK + tid * VE);
#pragma unroll
    for (int m = 0; m < NKQ; ++m) {
      const int e = tid + m * kThreads;
      const int arr = e / (kWin * KPR), rem = e % (kWin * KPR);
      const int tok = rem / KPR, pc = rem % KPR;
      if (tok < nt) {
        const size_t src = (size_t(w0 + tok) * Hl + h) * kDK + pc * VE;
        if (arr) cp_async16(&q[tok][pc * VE], qg + src);
        else cp_async16(&k[tok][pc * VE], kg + src);
      }
    }
#pragma unroll
    for (int m = 0; m < NV; ++m) {
      const int e = tid + m * kThreads;
      const int tok = e / VPR, pc = e % VPR, col = j0 + pc * VE;
      if (tok < nt && col < dv)
        cp_async16(&v[tok][pc * VE], vg + (size_t(w0 + tok) * Hl + h) * dv + col);
    }
    if (tid < kWin && tid < nt) cp_async4(&g[0][tid], alpha + size_t(w0 + tid) * Hl + h);
    if (tid >= kWin && tid < 2 * kWin && tid - kWin < nt)
      cp_async4(&g[1][tid - kWin], beta + size_t(w0 + tid - kWin) * Hl + h);
    cp_async_commit();
  }

  // 16 bytes as stored -> fp32 values at dst (bf16 widens exactly)
  __device__ __forceinline__ static void put(float* dst, const T* src) {
    const uint4 x = *reinterpret_cast<const uint4*>(src);
    if constexpr (sizeof(T) == 4) {
      *reinterpret_cast<uint4*>(dst) = x;
    } else {
      *reinterpret_cast<float4*>(dst) =
          make_float4(__uint_as_float(x.x << 16), __uint_as_float(x.x & 0xffff0000u),
                      __uint_as_float(x.y << 16), __uint_as_float(x.y & 0xffff0000u));
      *reinterpret_cast<float4*>(dst + 4) =
          make_float4(__uint_as_float(x.z << 16), __uint_as_float(x.z & 0xffff0000u),
                      __uint_as_float(x.w << 16), __uint_as_float(x.w & 0xffff0000u));
    }
  }

  // widen the landed window into the token loop's buffers (the extra k row
  // is zero when the prefix ends in this window)
  __device__ __forceinline__ void widen(float (*fk)[kPad], float (*fq)[kPad], float (*fv)[kCols],
                                        float* fa, float* fb, int nk, int tid) const {
    if (tid < KPR) {
      float* dst = fk[kWin] + padded(tid * VE);
      if (kWin < nk) {
        put(dst, &k[kWin][tid * VE]);
      } else {
#pragma unroll
        for (int x = 0; x < VE; x += 4)
          *reinterpret_cast<float4*>(dst + x) = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
#pragma unroll
    for (int m = 0; m < NKQ; ++m) {
      const int e = tid + m * kThreads;
      const int arr = e / (kWin * KPR), rem = e % (kWin * KPR);
      const int tok = rem / KPR, pc = rem % KPR;
      put((arr ? fq : fk)[tok] + padded(pc * VE), arr ? &q[tok][pc * VE] : &k[tok][pc * VE]);
    }
#pragma unroll
    for (int m = 0; m < NV; ++m) {
      const int e = tid + m * kThreads;
      put(fv[e / VPR] + (e % VPR) * VE, &v[e / VPR][(e % VPR) * VE]);
    }
    if (tid < kWin) fa[tid] = g[0][tid];
    else if (tid < 2 * kWin) fb[tid - kWin] = g[1][tid - kWin];
  }
};

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
    if (DELTA && w0 == p0) {
      // u of the prefix's first token, from the initial state
      float2 u0 = u, u1 = u;
#pragma unroll
      for (int m = 0; m < kRows / 4; ++m) {
        const float4 k4 = *reinterpret_cast<const float4*>(&fk[0][rb + 4 * m]);
        u0.x = fmaf(k4.x, s[4 * m].x, u0.x);     u0.y = fmaf(k4.x, s[4 * m].y, u0.y);
        u1.x = fmaf(k4.y, s[4 * m + 1].x, u1.x); u1.y = fmaf(k4.y, s[4 * m + 1].y, u1.y);
        u0.x = fmaf(k4.z, s[4 * m + 2].x, u0.x); u0.y = fmaf(k4.z, s[4 * m + 2].y, u0.y);
        u1.x = fmaf(k4.w, s[4 * m + 3].x, u1.x); u1.y = fmaf(k4.w, s[4 * m + 3].y, u1.y);
      }
      u = pair_sum_all(make_float2(u0.x + u1.x, u0.y + u1.y));
      u = make_float2(G * u.x, G * u.y);
    }
    for (int t = 0; t < nt; ++t) {
      const float a = fa[t], bt = fb[t];
      const float2 vv = *reinterpret_cast<const float2*>(&fv[t][cw]);
      float2 w = make_float2(bt * (vv.x - a * u.x), bt * (vv.y - a * u.y));
      float Gn = G * a;
      if (Gn < kMinGain) {
        // rare: fold the gain into the state so that 1 / Gn stays finite
        float f = G;
        Gn = a;
        if (a < kMinGain) {
          f = G * a;
          Gn = 1.f;
        }
#pragma unroll
        for (int i = 0; i < kRows; ++i) s[i] = make_float2(f * s[i].x, f * s[i].y);
      }
      // S' = Gn (s + k (w / Gn)^T); an approximate reciprocal only rescales
      // this token's rank-one term by a relative 2^-23 at most
      float ig;
      asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(ig) : "f"(Gn));
      w = make_float2(w.x * ig, w.y * ig);
      G = Gn;
      float2 op, un;
      // the next token's k is the staged row t + 1 (zero past the prefix)
      sweep<DELTA>(s, &fk[t][rb], &fq[t][rb], &fk[t + 1][rb], w, op, un);
      if (DELTA) {
        un = pair_sum_all(un);
        u = make_float2(G * un.x, G * un.y);
      }
      const float z = pair_sum_one(op, lane);
      if (writer) out[size_t(t) * out_step] = from_f32<T>(z * G * rs);
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
