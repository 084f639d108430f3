// Prefix scan of a linear-attention layer's recurrent state in chunks on the
// 5th-generation tensor cores (Sec. 4.1: the prefix state is computed once and
// every candidate forks from it). The recurrence is the one of the fork:
//   S_t = a_t (S_{t-1} - b_t k_t (k_t^T S_{t-1})) + b_t k_t v_t^T,
//   o_t = S_t^T q_t / sqrt(dk)                    (gated delta rule)
// or S_t = a_t S_{t-1} + b_t k_t v_t^T (plain gated linear attention).
//
// Over a chunk of C = 64 tokens starting from S0, with the decay products
// g_r = a_0 ... a_r and G[r][i] = a_{i+1} ... a_r (i <= r), the state after
// token r is S_r = g_r S0 + sum_{i<=r} G[r][i] k_i d_i^T, where the d_i solve
//   d_r + b_r sum_{i<r} G[r][i] (k_r . k_i) d_i = b_r v_r - b_r g_r S0^T k_r
// (d_r = b_r v_r for gated linear attention). Writing the solution of
// (I + A) X = B with A[r][i] = b_r G[r][i] (k_r . k_i) (i < r) for
// B = diag(b) V and B = diag(b g) K as U and W gives d = U - W S0, so
//   O   = diag(g) Q S0 + (M o G) d,  M[r][i] = q_r . k_i (i <= r)
//   S_C = g_{C-1} S0 + K^T diag(G[C-1][.]) d.
// Per chunk: one MMA gives [K; Q] K^T (the k.k and q.k products, exact in
// float32 from bf16 inputs); T = (I + A)^{-1} is formed on the CUDA cores in
// 16 x 16 blocks (the diagonal blocks by substitution, the rest as small
// products, level by level); then, on the transposed state (TMEM lane = value
// column):
//   U^T = V^T (T diag(b))^T,  W^T = K^T (T diag(b g))^T
//   X   = U^T + S0^T [-W | g Q]   -> d^T and (g Q S0)^T
//   X  += d^T (M o G)^T           -> O^T (accumulated onto (g Q S0)^T)
//   Dst = g_{C-1} S0^T + (d G[C-1])^T K  -> the next S0^T
// Operands that are not bf16 (S0, T diag(.), W, g Q, d, M o G) enter the MMA
// as a sum of two bf16 numbers (hi + lo, hi = bf16(x), lo = bf16(x - hi)): the
// products hi.hi + hi.lo + lo.hi keep about 16 bits, so the state keeps
// float32-like accuracy over the whole prefix. Forming T costs 64^3 / 6 FMAs a
// chunk instead of the 64^2 / 2 per column of a substitution for all 256
// columns of U and W.
//
// One CTA per (request, head); 8 warps: lane c of TMEM (value column c, and
// key column c of W) belongs to thread c of each warpgroup, which split the
// per-column work between them; thread 0 issues the MMAs and the TMA copies.
// The next chunk's K goes into a second buffer while the current chunk runs;
// Q and V are refilled as soon as the current chunk no longer reads them.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "jet_device.cuh"
#include "jet_internal.h"
#include "sm100_ptx.cuh"

namespace jet {
namespace {

using namespace sm100;

constexpr int kC = 64;         // tokens per chunk
constexpr int kD = 128;        // dk = dv handled by this kernel
constexpr int kThreads = 256;
constexpr uint64_t kDrainNs = 200000000ull;

// Shared memory (offsets from the 1024-byte aligned base). Operand tiles are
// K-major with 128-byte swizzling: 64 elements (128 bytes) per row, 8-row
// atoms of 1024 bytes, the 128-element dimension split into two slices.
// Each dk-slice of the token tiles holds [K buffer 0 | Q | K buffer 1] (64
// token rows each), so [K0; Q] (even chunks) and [Q; K1] (odd chunks) are
// 128-row operands.
constexpr uint32_t kKQSlice = 3 * 8192;
constexpr uint32_t kOffKQ = 0;
constexpr uint32_t kOffV = 2 * kKQSlice;            // V: 64 rows x 2 dv-slices
constexpr uint32_t kVSlice = 8192;
// 65536 .. 131071: free (the state's hi/lo operand lives in TMEM)
// [-W | g Q] hi, lo: MN-major (dk rows of 64 tokens), two N slices (-W, then
// g Q) of 128 rows; the first slices hold T diag(b) and T diag(b g) until W
constexpr uint32_t kOffWQh = 131072, kOffWQl = 163840;
constexpr uint32_t kWQSlice = 16384;
// once the first state MMA has read [-W | g Q]: d^T and (d G[C-1])^T, hi and
// lo, 128 rows (value column) x 64 tokens each
constexpr uint32_t kOffDh = 131072, kOffDl = 147456, kOffDGh = 163840, kOffDGl = 180224;
constexpr uint32_t kOffMh = 196608;     // (M o G) hi, lo: 64 rows (output token) x 64 tokens
constexpr uint32_t kOffMl = 204800;
constexpr uint32_t kOffA = 212992;      // A of the solve, 64 x 64 f32 (a_off)
constexpr uint32_t kOffVec = 229376;    // a[64], b[64], g[64], G[C-1][64], g_{C-1}
constexpr uint32_t kOffBar = kOffVec + 4 * 64 * 4 + 64;
constexpr uint32_t kSmemBytes = kOffBar + 64 + 1024;
static_assert(kSmemBytes <= 232448, "shared memory of one CTA");

// TMEM columns: [K; Q] K^T at 0 (64), X = [d^T | O^T] at 64 (128), the state
// at 256 (128), the state's hi and lo bf16 operand at 384 and 448 (64 each)
constexpr uint32_t kColGM = 0, kColX = 64, kColO = 128, kColSt = 256;
// the state as the X MMA's A operand: bf16 pairs (dk elements 2k, 2k + 1 of
// lane c in column k), hi then lo
constexpr uint32_t kColS0h = 384, kColS0l = 448;

// byte offset of element (row, k) in a 128-byte swizzled K-major tile
__device__ __forceinline__ uint32_t sw_off(int row, int k, uint32_t slice_bytes) {
  return uint32_t(k >> 6) * slice_bytes + uint32_t(row >> 3) * 1024u + uint32_t(row & 7) * 128u +
         (uint32_t(((k & 63) >> 3) ^ (row & 7)) << 4) + uint32_t(k & 7) * 2u;
}

// byte offset of the 16-byte chunk j (elements 8 j .. 8 j + 7) of a row
__device__ __forceinline__ uint32_t sw_chunk(int row, int j) {
  return uint32_t(row >> 3) * 1024u + uint32_t(row & 7) * 128u + (uint32_t(j ^ (row & 7)) << 4);
}

__device__ __forceinline__ float bf(const uint8_t* base, uint32_t off) {
  return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(base + off));
}

// x = hi + lo with hi, lo bf16
__device__ __forceinline__ void split2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  const float2 hf = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x - hf.x, y - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// 32 consecutive state values of this thread's lane (dk i0 .. i0 + 31) as hi
// and lo bf16 pairs in 16 TMEM columns each
__device__ __forceinline__ void put32_tmem(uint32_t hi_col, uint32_t lo_col, const float* x) {
  float h[16], l[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    uint32_t hh, ll;
    split2(x[2 * k], x[2 * k + 1], hh, ll);
    h[k] = __uint_as_float(hh);
    l[k] = __uint_as_float(ll);
  }
  tmem_st_16cols(hi_col, h);
  tmem_st_16cols(lo_col, l);
}

// eight consecutive values (chunk j of a 64-element slice row) as hi and lo
__device__ __forceinline__ void put8(uint8_t* hi_tile, uint8_t* lo_tile, int row, int j,
                                     const float* x) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) split2(x[2 * p], x[2 * p + 1], h[p], l[p]);
  const uint32_t off = sw_chunk(row, j);
  *reinterpret_cast<uint4*>(hi_tile + off) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo_tile + off) = make_uint4(l[0], l[1], l[2], l[3]);
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int32_t x, int32_t y, int32_t z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)),
      "l"(policy)
      : "memory");
}

// every thread waits (bounded); true when all of them saw the phase complete
__device__ __forceinline__ bool all_wait(uint64_t* bar, uint32_t par, uint64_t ns) {
  const bool ok = mbar_wait(bar, par, ns, nullptr);
  return __syncthreads_and(ok) != 0;
}

// A[r][i] (i < r) of the solve, row-major in f32 (a float index), the 16-byte
// chunks of row r permuted by r & 15 so that the rows written by consecutive
// threads fall in different banks; readers broadcast one chunk to the warp
__device__ __forceinline__ uint32_t a_off(int r, int chunk) {
  return uint32_t(r) * kC + (uint32_t(chunk ^ (r & 15)) << 2);
}

// T = (I + A)^{-1} (unit lower triangular) in f32, 64 floats a row, in the
// token tiles' two 8 KB Q slots (rows 32 s .. 32 s + 31 in slice s): the Q of
// the chunk is no longer needed when it is formed. Element (r, col): the
// 16-byte chunks of row r permuted by r & 15, so that the rows one warp
// reads or writes at the same columns fall in different banks.
__device__ __forceinline__ float* t_at(uint8_t* sm, int r, int col) {
  return reinterpret_cast<float*>(sm + kOffKQ + (r >> 5) * kKQSlice + 8192 + (r & 31) * 256 +
                                  ((((col >> 2) ^ (r & 15)) << 4) | ((col & 3) << 2)));
}

// T in 16 x 16 blocks: the diagonal blocks T_ii by substitution (thread
// (i, j): column j of T_ii) and, in the same step, the products T_ii A_ik
// (k < i) by substitution too, in the unused blocks above the diagonal; then
// the blocks below the diagonal level by level (d = i - j = 1, 2, 3):
// T_ij = -sum_{k=j}^{i-1} (T_ii A_ik) T_kj - four barrier-separated steps. Every block of T at or below the diagonal is
// written (zeros above the diagonal of T_ii). In the block products a thread
// forms four adjacent outputs of one row from 16-byte loads.
__device__ __forceinline__ void invert_unit_lower(const float* __restrict__ A, uint8_t* sm,
                                                  int tid) {
  if (tid < 64) {
    const int bi = tid >> 4, jj = tid & 15;
    float x[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      float s = r == jj ? 1.f : 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (4 * q < r) {
          const float4 a4 = *reinterpret_cast<const float4*>(A + a_off(16 * bi + r, 4 * bi + q));
          const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if (4 * q + e < r) s = fmaf(-av[e], x[4 * q + e], s);
        }
      }
      x[r] = s;
    }
#pragma unroll
    for (int r = 0; r < 16; ++r) *t_at(sm, 16 * bi + r, 16 * bi + jj) = x[r];
  } else if (tid < 64 + 6 * 16) {
    // in the same step, the six products T_ii A_ik (k < i), column by column as
    // the solutions of (I + A_ii) x = A_ik[:, col], each kept in the unused
    // block (k, i) above the diagonal
    const int task = tid - 64, b = task >> 4, col = task & 15;
    const int ib = b < 1 ? 1 : b < 3 ? 2 : 3, kb = b - ib * (ib - 1) / 2;
    float x[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      float s = A[a_off(16 * ib + r, 4 * kb + (col >> 2)) + (col & 3)];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        if (4 * q < r) {
          const float4 a4 = *reinterpret_cast<const float4*>(A + a_off(16 * ib + r, 4 * ib + q));
          const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if (4 * q + e < r) s = fmaf(-av[e], x[4 * q + e], s);
        }
      }
      x[r] = s;
    }
#pragma unroll
    for (int r = 0; r < 16; ++r) *t_at(sm, 16 * kb + r, 16 * ib + col) = x[r];
  }
  __syncthreads();
  // then the blocks below the diagonal level by level (d = i - j = 1, 2, 3):
  // T_ij = -sum_{k=j}^{i-1} (T_ii A_ik) T_kj, one barrier a level
#pragma unroll
  for (int d = 1; d < 4; ++d) {
    // task t: block (jb + d, jb), row r, columns 4 c4 .. 4 c4 + 3
    const int t = tid;
    const int jb = t >> 6, ib = jb + d, r = (t >> 2) & 15, c4 = t & 3;
    if (t < (4 - d) * 64) {
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      // 4 d chunks of k (a compile-time count: the loads can all be issued early)
#pragma unroll
      for (int kk = 0; kk < 4 * d; ++kk) {
        const int kb = jb + (kk >> 2), k4 = kk & 3;
        const float4 p4 = *reinterpret_cast<const float4*>(t_at(sm, 16 * kb + r, 16 * ib + 4 * k4));
        const float pv[4] = {p4.x, p4.y, p4.z, p4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float4 t4 =
              *reinterpret_cast<const float4*>(t_at(sm, 16 * kb + 4 * k4 + e, 16 * jb + 4 * c4));
          acc.x = fmaf(pv[e], t4.x, acc.x);
          acc.y = fmaf(pv[e], t4.y, acc.y);
          acc.z = fmaf(pv[e], t4.z, acc.z);
          acc.w = fmaf(pv[e], t4.w, acc.w);
        }
      }
      *reinterpret_cast<float4*>(t_at(sm, 16 * ib + r, 16 * jb + 4 * c4)) =
          make_float4(-acc.x, -acc.y, -acc.z, -acc.w);
    }
    __syncthreads();
  }
}

template <bool DELTA>
__global__ void __launch_bounds__(kThreads, 1)
scan_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, const int32_t* __restrict__ prefix_offset,
               int R, int total, int Hl, const float* __restrict__ s_init,
               const float* __restrict__ alpha, const float* __restrict__ beta,
               __nv_bfloat16* __restrict__ o, float* __restrict__ s_out, int* status,
               uint64_t wait_ns, int hold_first) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                           ~uintptr_t(1023));
  float* va = reinterpret_cast<float*>(sm + kOffVec);  // a of the chunk's tokens (1 past its end)
  float* vb = va + 64;                                 // b (0 past its end)
  float* vg = vb + 64;                                 // g_r = a_0 ... a_r
  float* vgc = vg + 64;                                // G[C-1][i]
  float* gC = vgc + 64;                                // g_{C-1}
  float* Am = reinterpret_cast<float*>(sm + kOffA);
  // the chunk's outputs [64 tokens][kD] bf16, staged in the A buffer
  __nv_bfloat16* ost = reinterpret_cast<__nv_bfloat16*>(sm + kOffA);
  uint64_t* bar_k = reinterpret_cast<uint64_t*>(sm + kOffBar);  // K buffers 0 and 1
  uint64_t* bar_q = bar_k + 2;
  uint64_t* bar_v = bar_k + 3;
  uint64_t* bar_mma = bar_k + 4;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar_k + 5);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int grp = tid >> 7;   // warpgroup
  const int c = tid & 127;    // TMEM lane: value column c (and key column c of W)
  const int h = blockIdx.x, r = blockIdx.y;
  if (tid == 0) {
    for (int b = 0; b < 5; ++b) mbar_init(bar_k + b, 1);
    fence_barrier_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  pdl_begin();
  if (warp == 0) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  const uint32_t lane_off = uint32_t(32 * (warp & 3)) << 16;
  int p0 = 0, p1 = 0;
  if (r < R) {
    p0 = prefix_offset[r];
    p1 = prefix_offset[r + 1];
  }
  if (r >= R || p0 < 0 || p1 < p0 || p1 > total) {
    if (tid == 0) flag(status, JET_ERR_DEVICE);
    p1 = p0 = 0;
  }
  const int nch = (p1 - p0 + kC - 1) / kC;
  const size_t head = (size_t(r) * Hl + h) * kD;  // row 0 of this (request, head)'s state
  const uint64_t pol = policy_evict_first();

  // TMA copies of chunk j's K (into buffer j & 1), Q and V, issued by thread 0;
  // `pend` marks the barriers with a copy in flight (bits 0, 1: K buffers, 2:
  // Q, 3: V)
  uint32_t pend = 0;
  auto load_k = [&](int j) {
    uint64_t* b = bar_k + (j & 1);
    mbar_arrive_expect_tx(b, 2 * 8192);
    for (int sl = 0; sl < 2; ++sl)
      tma_load_3d(sm + kOffKQ + sl * kKQSlice + (j & 1) * 16384, &tmK, b, sl * 64, h,
                  p0 + j * kC, pol);
    pend |= 1u << (j & 1);
  };
  auto load_q = [&](int j) {
    mbar_arrive_expect_tx(bar_q, 2 * 8192);
    for (int sl = 0; sl < 2; ++sl)
      tma_load_3d(sm + kOffKQ + sl * kKQSlice + 8192, &tmQ, bar_q, sl * 64, h, p0 + j * kC, pol);
    pend |= 4u;
  };
  auto load_v = [&](int j) {
    mbar_arrive_expect_tx(bar_v, 2 * 8192);
    for (int sl = 0; sl < 2; ++sl)
      tma_load_3d(sm + kOffV + sl * kVSlice, &tmV, bar_v, sl * 64, h, p0 + j * kC, pol);
    pend |= 8u;
  };
  if (tid == 0 && nch > 0 && !hold_first) {
    load_k(0);
    load_q(0);
    load_v(0);
    if (nch > 1) load_k(1);
  }
  // the gates of the first chunk (thread t < 64: token t of the chunk)
  float na = 1.f, nb = 0.f;
  if (tid < kC && p0 + tid < p1) {
    na = alpha[size_t(p0 + tid) * Hl + h];
    nb = beta[size_t(p0 + tid) * Hl + h];
  }

  // the initial state: into TMEM (lane c holds S0^T[c][.] = S0[.][c]; this
  // warpgroup's 64 columns) and as the bf16 hi/lo operand of the first state MMA
  for (int i0 = 64 * grp; i0 < 64 * grp + 64; i0 += 32) {
    float v[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = s_init ? s_init[(head + i0 + i) * kD + c] : 0.f;
    tmem_st_32cols(tmem + lane_off + kColSt + i0, v);
    put32_tmem(tmem + lane_off + kColS0h + (i0 >> 1), tmem + lane_off + kColS0l + (i0 >> 1), v);
  }
  tmem_wait_st();
  fence_proxy_async_shared();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  const float rs = rsqrtf(float(kD));
  uint32_t kph = 0, qph = 0, vph = 0, mph = 0;  // kph: bit b = parity of K buffer b
  bool ok = true;
  for (int j = 0; ok && j < nch; ++j) {
    const int c0 = p0 + j * kC;
    const int n = min(kC, p1 - c0);
    const bool last = j + 1 == nch;
    const int odd = j & 1;
    uint8_t* const kt = sm + kOffKQ + odd * 16384;  // this chunk's K (dk-slices kKQSlice apart)
    // ---- gates and decay products
    if (tid < kC) {
      va[tid] = na;
      vb[tid] = nb;
    }
    __syncthreads();
    if (tid < kC && !last) {
      const int t = c0 + kC + tid;
      na = t < p1 ? alpha[size_t(t) * Hl + h] : 1.f;
      nb = t < p1 ? beta[size_t(t) * Hl + h] : 0.f;
    }
    // row rr (first warpgroup): G[rr][i] = a_{i+1} .. a_rr (i <= rr), g_rr
    const int rr = tid & 63;
    float gam[kC];
    if (grp == 0) {
      float g = 1.f;
#pragma unroll
      for (int i = kC - 1; i >= 0; --i) {
        gam[i] = i <= rr ? g : 0.f;
        if (i <= rr) g *= va[i];
      }
      if (tid < kC) vg[rr] = g;
      if (tid == kC - 1) {
        *gC = g;
#pragma unroll
        for (int i = 0; i < kC; ++i) vgc[i] = gam[i];
      }
    }
    {
      const bool okk = mbar_wait(bar_k + odd, (kph >> odd) & 1u, wait_ns, nullptr) &&
                       mbar_wait(bar_q, qph, wait_ns, nullptr);
      ok = __syncthreads_and(okk) != 0;
    }
    if (!ok) break;
    kph ^= 1u << odd;
    qph ^= 1u;
    if (tid == 0) pend &= ~((1u << odd) | 4u);
    // ---- [K; Q] K^T (even chunks) or [Q; K] K^T (odd): k.k and q.k in float32
    if (tid == 0) {
      tc_fence_after();
#pragma unroll
      for (int st = 0; st < 8; ++st) {
        const uint32_t sl = (st >> 2) * kKQSlice + 32 * (st & 3);
        const uint32_t a = smem_u32(sm + kOffKQ + (odd ? 8192 : 0)) + sl;
        const uint32_t b = smem_u32(kt) + sl;
        mma_f16(tmem + kColGM, desc_k_sw128(a), desc_k_sw128(b), idesc_bf16_f32(128, 64), st != 0);
      }
      mma_commit(bar_mma);
    }
    ok = all_wait(bar_mma, mph, wait_ns);
    if (!ok) break;
    mph ^= 1u;
    tc_fence_after();
    // ---- the solve's matrix A (k rows) and M o G (q rows) from the first
    // warpgroup's TMEM lanes; g Q from the second warpgroup
    if (grp == 0) {
      // 32 columns of [K; Q] K^T at a time
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        float gr[32];
        tmem_ld_32cols(tmem + lane_off + kColGM + 32 * hf, gr);
        tmem_wait_ld();
        if ((tid >> 6) == odd) {
          // k row rr: A[rr][i] = b_rr G[rr][i] (k_rr . k_i), i < rr (the
          // entries from rr on are never read)
          if (DELTA) {
            const float b = vb[rr];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const int i = 32 * hf + 4 * q;
              float4 w;
              w.x = i + 0 < rr ? b * gam[i + 0] * gr[4 * q + 0] : 0.f;
              w.y = i + 1 < rr ? b * gam[i + 1] * gr[4 * q + 1] : 0.f;
              w.z = i + 2 < rr ? b * gam[i + 2] * gr[4 * q + 2] : 0.f;
              w.w = i + 3 < rr ? b * gam[i + 3] * gr[4 * q + 3] : 0.f;
              *reinterpret_cast<float4*>(Am + a_off(rr, 8 * hf + q)) = w;
            }
          }
        } else {
          // q row rr: (M o G)[rr][i] = (q_rr . k_i) G[rr][i], i <= rr
          float m[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) m[i] = gam[32 * hf + i] * gr[i];  // gam = 0 past rr
#pragma unroll
          for (int jj = 0; jj < 4; ++jj)
            put8(sm + kOffMh, sm + kOffMl, rr, 4 * hf + jj, m + 8 * jj);
        }
      }
    } else {
      // g Q as rows 64 .. 127 (the second N slice) of the MN-major [-W | g Q]
      // operand: thread c writes dk row c, the chunk's 64 tokens contiguous
      const uint8_t* qt = sm + kOffKQ + 8192;
      float x[kC];
#pragma unroll
      for (int t = 0; t < kC; ++t) x[t] = vg[t] * bf(qt, sw_off(t, c, kKQSlice));
#pragma unroll
      for (int jj = 0; jj < 8; ++jj)
        put8(sm + kOffWQh + kWQSlice, sm + kOffWQl + kWQSlice, c, jj, x + 8 * jj);
      if (DELTA) {
        // O^T starts from zero under the first state MMA's accumulation
        float z[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) z[i] = 0.f;
        tmem_st_32cols(tmem + lane_off + kColO, z);
        tmem_st_32cols(tmem + lane_off + kColO + 32, z);
      }
    }
    tmem_wait_st();
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();
    if (DELTA) {
      // ---- T = (I + A)^{-1}, then T' = T diag(b) and T'' = T diag(b g) as
      // the hi/lo B operands (row r, 64 tokens i, K-major) of U = T' V and
      // W = T'' K, in the first N slice of the [-W | g Q] tiles (free until W)
      invert_unit_lower(Am, sm, tid);
      {
        const int row = tid >> 2;
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
          const int jj = 2 * (tid & 3) + h2;
          float x1[8], x2[8];
          const float4 t0 = *reinterpret_cast<const float4*>(t_at(sm, row, 8 * jj));
          const float4 t1 = *reinterpret_cast<const float4*>(t_at(sm, row, 8 * jj + 4));
          const float tv[8] = {t0.x, t0.y, t0.z, t0.w, t1.x, t1.y, t1.z, t1.w};
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int i = 8 * jj + e;
            const float t = i <= row ? tv[e] : 0.f;
            x1[e] = t * vb[i];
            x2[e] = x1[e] * vg[i];
          }
          put8(sm + kOffWQh, sm + kOffWQl, row, jj, x1);
          put8(sm + kOffWQh + 8192, sm + kOffWQl + 8192, row, jj, x2);
        }
      }
      fence_proxy_async_shared();
      tc_fence_before();
      __syncthreads();
    }
    // Q (and T in its slots) is no longer read: the next chunk's Q may land
    if (tid == 0 && !last) load_q(j + 1);
    ok = all_wait(bar_v, vph, wait_ns);
    if (!ok) break;
    vph ^= 1u;
    if (tid == 0) pend &= ~8u;
    if (DELTA) {
      // ---- U^T = V^T T'^T (TMEM at X, for the first state MMA to accumulate
      // onto) and W^T = K^T T''^T: V and K are MN-major A operands (exact in
      // bf16), T' and T'' enter as hi + lo
      if (tid == 0) {
        tc_fence_after();
        const uint32_t idesc = idesc_bf16_f32(128, 64) | (1u << 15);
#pragma unroll
        for (int pass = 0; pass < 2; ++pass) {
          const uint32_t b = smem_u32(sm + (pass ? kOffWQl : kOffWQh));
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            mma_f16(tmem + kColX, desc_mn_sw128(smem_u32(sm + kOffV) + k * 2048, kVSlice),
                    desc_k_sw128(b + 32 * k), idesc, (pass | k) != 0);
            mma_f16(tmem + kColGM, desc_mn_sw128(smem_u32(kt) + k * 2048, kKQSlice),
                    desc_k_sw128(b + 8192 + 32 * k), idesc, (pass | k) != 0);
          }
        }
        mma_commit(bar_mma);
      }
      ok = all_wait(bar_mma, mph, wait_ns);
      if (!ok) break;
      mph ^= 1u;
      tc_fence_after();
      // -W as the first N slice of [-W | g Q]: thread c writes key row c
      if (grp == 1) {
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          float wv[32];
          tmem_ld_32cols(tmem + lane_off + kColGM + 32 * hf, wv);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) wv[i] = -wv[i];
#pragma unroll
          for (int jj = 0; jj < 4; ++jj)
            put8(sm + kOffWQh, sm + kOffWQl, c, 4 * hf + jj, wv + 8 * jj);
        }
      }
    } else if (grp == 0) {
      // gated linear attention: U = diag(b) V straight into TMEM
      const uint8_t* vt = sm + kOffV;
#pragma unroll
      for (int i0 = 0; i0 < kC; i0 += 32) {
        float uv[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) uv[i] = vb[i0 + i] * bf(vt, sw_off(i0 + i, c, kVSlice));
        tmem_st_32cols(tmem + lane_off + kColX + i0, uv);
      }
      tmem_wait_st();
    }
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();
    // V is no longer read
    if (tid == 0 && !last) load_v(j + 1);
    // ---- X = U^T + S0^T [-W | g Q] (delta rule) or O^T = S0^T (g Q)
    // (gated linear attention, X = U^T as stored): three hi/lo passes; the B
    // operand is MN-major (dk rows of 128 tokens)
    if (tid == 0) {
      tc_fence_after();
#pragma unroll
      for (int pass = 0; pass < 3; ++pass) {
        // A (the state, K = dk) from TMEM: 8 packed columns per K = 16 step
        const uint32_t a = tmem + (pass == 2 ? kColS0l : kColS0h);
        const uint32_t b = smem_u32(sm + (pass == 1 ? kOffWQl : kOffWQh));
#pragma unroll
        for (int st = 0; st < 8; ++st) {
          if (DELTA)
            mma_f16_ta(tmem + kColX, a + 8 * st, desc_mn_sw128(b + st * 2048, kWQSlice),
                       idesc_bf16_f32(128, 128) | (1u << 16), 1u);
          else
            mma_f16_ta(tmem + kColO, a + 8 * st, desc_mn_sw128(b + kWQSlice + st * 2048, kWQSlice),
                       idesc_bf16_f32(128, 64) | (1u << 16), (pass | st) != 0);
        }
      }
      mma_commit(bar_mma);
    }
    ok = all_wait(bar_mma, mph, wait_ns);
    if (!ok) break;
    mph ^= 1u;
    tc_fence_after();
    // ---- d (column c of d is row c of d^T): the first warpgroup writes d^T,
    // the second (d G[C-1])^T, as the second MMA group's A operands; each
    // scales its 64 state columns by g_{C-1} in TMEM for the last MMA to
    // accumulate onto
    {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        float dr[32];
        tmem_ld_32cols(tmem + lane_off + kColX + 32 * hf, dr);
        tmem_wait_ld();
        if (grp == 0) {
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) put8(sm + kOffDh, sm + kOffDl, c, 4 * hf + jj, dr + 8 * jj);
        } else {
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) {
            float dg[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) dg[e] = dr[8 * jj + e] * vgc[32 * hf + 8 * jj + e];
            put8(sm + kOffDGh, sm + kOffDGl, c, 4 * hf + jj, dg);
          }
        }
      }
      const float g = *gC;
      const uint32_t scol = tmem + lane_off + kColSt + 64 * grp;
      float s0[32], s1[32];
      tmem_ld_32cols(scol, s0);
      tmem_ld_32cols(scol + 32, s1);
      tmem_wait_ld();
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        s0[i] *= g;
        s1[i] *= g;
      }
      tmem_st_32cols(scol, s0);
      tmem_st_32cols(scol + 32, s1);
      tmem_wait_st();
    }
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();
    // ---- O^T += d^T (M o G)^T (three passes); state^T += (d G[C-1])^T K (two:
    // K is exact in bf16)
    if (tid == 0) {
      tc_fence_after();
#pragma unroll
      for (int pass = 0; pass < 3; ++pass) {
        const uint32_t a = smem_u32(sm + (pass == 2 ? kOffDl : kOffDh));
        const uint32_t b = smem_u32(sm + (pass == 1 ? kOffMl : kOffMh));
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_f16(tmem + kColO, desc_k_sw128(a + 32 * k), desc_k_sw128(b + 32 * k),
                  idesc_bf16_f32(128, 64), 1u);
      }
#pragma unroll
      for (int pass = 0; pass < 2; ++pass) {
        const uint32_t a = smem_u32(sm + (pass == 1 ? kOffDGl : kOffDGh));
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_f16(tmem + kColSt, desc_k_sw128(a + 32 * k),
                  desc_mn_sw128(smem_u32(kt) + k * 16 * 128, kKQSlice),
                  idesc_bf16_f32(128, 128) | (1u << 16), 1u);
      }
      mma_commit(bar_mma);
    }
    ok = all_wait(bar_mma, mph, wait_ns);
    if (!ok) break;
    mph ^= 1u;
    tc_fence_after();
    // this chunk's K is no longer read: the chunk after next may land there
    if (tid == 0 && j + 2 < nch) load_k(j + 2);
    // ---- outputs of the chunk's tokens (warpgroup g: tokens 32 g ..), and this
    // warpgroup's 64 columns of the new state as the next chunk's operand (and,
    // after the last chunk, the result)
    {
      float ov[32];
      tmem_ld_32cols(tmem + lane_off + kColO + 32 * grp, ov);
      const uint32_t scol = tmem + lane_off + kColSt + 64 * grp;
      float s0[32], s1[32];
      tmem_ld_32cols(scol, s0);
      tmem_ld_32cols(scol + 32, s1);
      tmem_wait_ld();
      // the chunk's outputs through the solve's A buffer (free until the next
      // chunk), [token][value] as they are stored, for 16-byte global stores
#pragma unroll
      for (int i = 0; i < 32; ++i) ost[(32 * grp + i) * kD + c] = __float2bfloat16_rn(ov[i] * rs);
      if (last) {
        const size_t row0 = head + 64 * grp;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          s_out[(row0 + i) * kD + c] = s0[i];
          s_out[(row0 + 32 + i) * kD + c] = s1[i];
        }
      } else {
        // this warpgroup's 64 dk columns: packed columns 32 grp .. 32 grp + 31
        put32_tmem(tmem + lane_off + kColS0h + 32 * grp, tmem + lane_off + kColS0l + 32 * grp, s0);
        put32_tmem(tmem + lane_off + kColS0h + 32 * grp + 16,
                   tmem + lane_off + kColS0l + 32 * grp + 16, s1);
        tmem_wait_st();
      }
    }
    fence_proxy_async_shared();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // each token's 128 outputs are 256 contiguous bytes of o (the next
    // chunk's first barrier comes before its A lands in the buffer)
    for (int e = tid; e < n * (kD / 8); e += kThreads) {
      const int t = e / (kD / 8), q = e % (kD / 8);
      *reinterpret_cast<uint4*>(o + (size_t(c0 + t) * Hl + h) * kD + 8 * q) =
          reinterpret_cast<const uint4*>(ost)[e];
    }
  }
  if (!ok) {
    // a wait ran out: let the copies and tensor-core work already issued
    // finish before the CTA frees its TMEM and ends
    if (tid == 0) {
      flag(status, JET_ERR_TIMEOUT);
      for (int b = 0; b < 2; ++b)
        if (pend & (1u << b)) mbar_wait(bar_k + b, (kph >> b) & 1u, kDrainNs, nullptr);
      if (pend & 4u) mbar_wait(bar_q, qph, kDrainNs, nullptr);
      if (pend & 8u) mbar_wait(bar_v, vph, kDrainNs, nullptr);
      mma_commit(bar_mma);
      mbar_wait(bar_mma, mph, kDrainNs, nullptr);
    }
  } else if (p1 == p0 && r < R && s_out != nullptr) {
    // no prefix tokens: the state is the initial one (zeros without one)
    for (int i = 64 * grp; i < 64 * grp + 64; ++i)
      s_out[(head + i) * kD + c] = s_init ? s_init[(head + i) * kD + c] : 0.f;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// [tokens, Hl, 128] bf16: boxes of 64 elements x 1 head x 64 tokens, 128-byte swizzle
bool encode_tokens(CUtensorMap* map, const void* base, int tokens, int Hl) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {cuuint64_t(kD), cuuint64_t(Hl), cuuint64_t(tokens)};
  const cuuint64_t strides[2] = {cuuint64_t(kD) * 2, cuuint64_t(Hl) * kD * 2};
  const cuuint32_t box[3] = {64, 1, cuuint32_t(kC)};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool scan_tc_supported(const jet_dims& d) {
  return d.dtype == JET_DTYPE_BF16 && d.dk == kD && d.dv == kD;
}

cudaError_t launch_scan_tc(const jet_layout& lay, const jet_dims& d, int rule,
                           const float* s_init, const void* q, const void* k, const void* v,
                           const float* alpha, const float* beta, void* o, float* s_out,
                           int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  CUtensorMap tmQ, tmK, tmV;
  if (!encode_tokens(&tmQ, q, n.total_prefix, d.Hl) ||
      !encode_tokens(&tmK, k, n.total_prefix, d.Hl) ||
      !encode_tokens(&tmV, v, n.total_prefix, d.Hl))
    return cudaErrorInvalidValue;
  auto kern = rule == JET_RECUR_GLA ? scan_tc_kernel<false> : scan_tc_kernel<true>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(unsigned(d.Hl), unsigned(n.R)), dim3(kThreads), kSmemBytes, st,
                    tmQ, tmK, tmV, lay.prefix_offset, n.R, n.total_prefix, d.Hl, s_init, alpha,
                    beta, static_cast<__nv_bfloat16*>(o), s_out, status, wait_budget_ns(),
                    test_stall());
}

}  // namespace jet
