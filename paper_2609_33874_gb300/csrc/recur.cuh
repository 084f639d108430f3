// Device code of the register-resident linear-attention recurrence (the
// prefix scan, scan.cu): a CTA keeps a
// 128 x 64 slice of the state S in registers (thread = 32 rows x 2 columns,
// the lanes of a row group adjacent), fed tokens are staged 16 at a time
// (asynchronous copies into a raw buffer, widened to fp32 at the window
// boundary, one extra k row for the window's last token), and one sweep over
// a thread's rows per token applies the update and accumulates the output and
// the next token's k^T S. Included inside an anonymous namespace.
#pragma once


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

// k^T S for the staged k row kr over this thread's rows (kr already offset to
// them), reduced over the column pair; G S~ = S
__device__ __forceinline__ float2 k_dot_s(const float2 (&s)[kRows], const float* kr, float G) {
  float2 u0 = make_float2(0.f, 0.f), u1 = u0;
#pragma unroll
  for (int m = 0; m < kRows / 4; ++m) {
    const float4 k4 = *reinterpret_cast<const float4*>(kr + 4 * m);
    u0.x = fmaf(k4.x, s[4 * m].x, u0.x);     u0.y = fmaf(k4.x, s[4 * m].y, u0.y);
    u1.x = fmaf(k4.y, s[4 * m + 1].x, u1.x); u1.y = fmaf(k4.y, s[4 * m + 1].y, u1.y);
    u0.x = fmaf(k4.z, s[4 * m + 2].x, u0.x); u0.y = fmaf(k4.z, s[4 * m + 2].y, u0.y);
    u1.x = fmaf(k4.w, s[4 * m + 3].x, u1.x); u1.y = fmaf(k4.w, s[4 * m + 3].y, u1.y);
  }
  const float2 u = pair_sum_all(make_float2(u0.x + u1.x, u0.y + u1.y));
  return make_float2(G * u.x, G * u.y);
}

// One token of the recurrence on this thread's slice of S = G s~:
// S <- alpha S + beta k (v - alpha u)^T with u = k^T S of the token (the
// delta rule; u = 0 for gated linear attention), then o = S^T q. kt, qt, kn
// are the token's staged k and q rows and the next token's k row (NEXT: u of
// the next token is computed in the same sweep). Returns this lane's column
// of o (unscaled by 1 / sqrt(dk)).
template <bool DELTA, bool NEXT>
__device__ __forceinline__ float recur_token(float2 (&s)[kRows], float& G, float2& u, float a,
                                             float bt, float2 vv, const float* kt,
                                             const float* qt, const float* kn, int lane) {
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
  // S' = Gn (s + k (w / Gn)^T); an approximate reciprocal only rescales this
  // token's rank-one term by a relative 2^-23 at most
  float ig;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(ig) : "f"(Gn));
  w = make_float2(w.x * ig, w.y * ig);
  G = Gn;
  float2 op, un;
  sweep<DELTA && NEXT>(s, kt, qt, kn, w, op, un);
  if (DELTA && NEXT) {
    un = pair_sum_all(un);
    u = make_float2(G * un.x, G * un.y);
  }
  return pair_sum_one(op, lane) * G;
}

