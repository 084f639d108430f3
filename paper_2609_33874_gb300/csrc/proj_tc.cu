// Projections of a decoder stack on the 5th-generation tensor cores:
// out[N, O] = epilogue(X[N, K] W[O, K]^T) with bf16 X and W and f32
// accumulation, for the mixer, output and MLP projections of every layer.
//
// Clusters of two CTAs (one per SM) work through units of (256 weight rows,
// one token tile of up to 256 of the step's rows, a K range): each CTA loads
// its own 128 weight rows and half of the token tile (the even CTA the first
// Nt / 2 rows) into a ring of stages, both CTAs' loads complete on the even
// CTA's stage barrier, and the even CTA issues M = 256 MMAs
// (tcgen05.mma.cta_group::2) whose products land in both CTAs' TMEM, each CTA
// holding its own 128 weight rows over all Nt columns. Per stage a CTA takes in
// 16 KB of weights and Nt x 64 bytes of rows for 128 x Nt outputs (alone it
// would take Nt x 128 bytes of rows): the tile bytes one SM takes in, not HBM,
// bound these small-N GEMMs.
//   warp 0      TMA producer (each CTA): its 128 x 64 weight tile and
//               Nt / 2 x 64 row tile per stage, both 128-byte swizzled
//   warp 1      TMEM allocator (each CTA, together) and, in the even CTA,
//               the MMA issuer: 4 x tcgen05.mma kind::f16 (K = 16) per stage
//               into one of two TMEM accumulators; the commits reach both
//               CTAs' barriers
//   warps 2..5  epilogue (each CTA): each warp reads its 32 TMEM lanes (32
//               output features) x 32 rows at a time and writes bf16 outputs
// Epilogues: kStore (out = acc), kResid (out = res + acc, one rounding; res
// may be out itself: every element is read and written by one thread) and
// kSwiGLU: the weight rows come interleaved in blocks of 64 (tile rows 0..63
// gate features 64 t .., rows 64..127 the matching up features), the halves
// exchange half of their columns through shared memory, and
// out[n, 64 t + f] = SiLU(gate) * up.
// Split K: when the units are too few to occupy the SM pairs (few output
// features, long K), each unit covers a range of K and writes its f32 partial;
// a reduce kernel sums the partials and applies the epilogue.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <mutex>

#include "jet_device.cuh"
#include "jet_internal.h"
#include "sm100_ptx.cuh"

namespace jet {
namespace {

using namespace sm100;

constexpr int kBM = 128;            // weight rows per CTA (MMA M per CTA, TMEM lanes)
constexpr int kBK = 64;             // bf16 elements per stage: 128 bytes
constexpr int kThreads = 192;
constexpr int kMaxNt = 256;
constexpr uint64_t kDrainNs = 200000000ull;
constexpr int kSmemLimit = 232448;
// gate/up exchange (16 columns x 128 lanes f32) + barriers and flags
constexpr int kFixedSmem = 16 * 128 * 4 + 32 * 8 + 64;

struct ProjArgs {
  __nv_bfloat16* out;
  const __nv_bfloat16* res;
  float* part;          // split K: f32 partials [splits][N][O]
  int* status;
  int N, O, K, ldo;     // rows, weight rows, reduction length, output row stride
  int Nt, n_tt, units, nkb, stages, splits;
  uint32_t tmem_cols, acc_cols;  // two accumulators of acc_cols columns
  uint64_t wait_ns;  // budget of one bounded wait (jet_set_wait_budget_ns)
  int hold_first;    // test hook (jet_set_test_stall): withhold the first stage's loads
  int vec;           // out 16-byte aligned and ldo % 8 == 0: 16-byte output stores
};

// unit u -> (256-row weight slice, K split, token tile); the token tiles of one
// weight slice are consecutive, so they share it through L2
struct Unit {
  int ot, sp, t0, kb0, kb1;
};
__device__ __forceinline__ Unit unit_of(const ProjArgs& a, int u) {
  Unit x;
  const int tt = u % a.n_tt, rest = u / a.n_tt;
  x.sp = rest % a.splits;
  x.ot = rest / a.splits;
  x.t0 = tt * a.Nt;
  x.kb0 = int((long long)x.sp * a.nkb / a.splits);
  x.kb1 = int((long long)(x.sp + 1) * a.nkb / a.splits);
  return x;
}

template <int EPI>
__global__ void __launch_bounds__(kThreads, 1)
proj_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
               const ProjArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t a_bytes = kBM * 128, b_bytes = uint32_t(a.Nt / 2) * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  float* upx = reinterpret_cast<float*>(smem + size_t(a.stages) * stage_bytes);  // [16][128]
  uint64_t* full = reinterpret_cast<uint64_t*>(upx + 16 * 128);
  uint64_t* empty = full + a.stages;
  uint64_t* tfull = empty + a.stages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* epi_abort = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // this CTA's rank in its pair, the pair's number and the number of pairs
  const uint32_t rank = cluster_rank();
  const int cid = int(blockIdx.x >> 1), ncl = int(gridDim.x >> 1);
  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, 8);  // both CTAs' epilogue warps
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    *epi_abort = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
  }
  pdl_begin();
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, a.tmem_cols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the even CTA's barriers are initialised before any remote use
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_x = policy_evict_last();
      int s = 0;
      uint32_t ph = 0, issued = 0, issued_par = 0;
      bool ok = true, hold = a.hold_first != 0;
      for (int u = cid; ok && u < a.units; u += ncl) {
        const Unit x = unit_of(a, u);
        const int o0 = (2 * x.ot + int(rank)) * kBM;
        const int t0 = x.t0 + int(rank) * (a.Nt / 2);
        for (int kb = x.kb0; kb < x.kb1; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1u, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + size_t(s) * stage_bytes;
          if (hold) {
            hold = false;  // test hook: this stage never fills
          } else {
            // both CTAs' bytes complete on the even CTA's barrier, which
            // expects them all; the odd CTA's may land before that arrive
            const uint32_t bar = mapa_shared(full + s, 0);
            if (rank == 0) mbar_arrive_expect_tx(full + s, 2 * stage_bytes);
            tma_load_2d_pair(sa, &tmW, bar, kb * kBK, o0, pol_w);
            tma_load_2d_pair(sa + a_bytes, &tmX, bar, kb * kBK, t0, pol_x);
            issued |= 1u << s;
            issued_par = (issued_par & ~(1u << s)) | (ph << s);
          }
          if (++s == a.stages) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        // let the copies in flight land: the even CTA's barriers count both
        // CTAs' bytes; the odd CTA waits out a fixed bounded time
        if (rank == 0) {
          for (int t = 0; t < a.stages; ++t)
            if (issued & (1u << t)) mbar_wait(full + t, (issued_par >> t) & 1u, kDrainNs, nullptr);
        } else if (issued) {
          const uint64_t t0 = global_timer_ns();
          while (global_timer_ns() - t0 < kDrainNs / 16) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && rank == 0) {
      const uint32_t idesc = idesc_bf16_f32(2 * kBM, a.Nt);
      int s = 0, local = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int u = cid; ok && u < a.units; u += ncl, ++local) {
        const int buf = local & 1;
        const uint32_t tph = (local >> 1) & 1;
        if (!mbar_wait(tempty + buf, tph ^ 1u, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + uint32_t(buf) * a.acc_cols;
        const Unit x = unit_of(a, u);
        for (int kb = x.kb0; kb < x.kb1; ++kb) {
          if (!mbar_wait(full + s, ph, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // one thread issues every MMA, so the loop stays lean: the
          // descriptors are built once per stage and stepped along K by
          // adding to their start-address field (16-byte units)
          const uint32_t sa = smem_u32(smem + size_t(s) * stage_bytes);
          const uint64_t da = desc_k_sw128(sa), db = desc_k_sw128(sa + a_bytes);
          mma_f16_pair(d_tmem, da, db, idesc, kb != x.kb0);
          mma_f16_pair(d_tmem, da + 2, db + 2, idesc, 1u);
          mma_f16_pair(d_tmem, da + 4, db + 4, idesc, 1u);
          mma_f16_pair(d_tmem, da + 6, db + 6, idesc, 1u);
          mma_commit_pair(empty + s, 0x3);  // both CTAs' stage s is free
          if (++s == a.stages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit_pair(tfull + buf, 0x3);
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        mma_commit_pair(drain, 0x1);
        mbar_wait(drain, 0, kDrainNs, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;            // TMEM lane quadrant this warp may access
    // the odd CTA's warps release the accumulator on the even CTA's barrier
    const uint32_t tempty_even = mapa_shared(tempty, 0);
    int local = 0;
    for (int u = cid; u < a.units; u += ncl, ++local) {
      const int buf = local & 1;
      const uint32_t tph = (local >> 1) & 1;
      const Unit x = unit_of(a, u);
      const int t0 = x.t0;
      const bool ok = warp_mbar_wait(tfull + buf, tph, a.wait_ns, abort_flag);
      if (!ok || *abort_flag) *epi_abort = 1;
      named_bar_sync(1, 128);
      if (*epi_abort) break;
      tc_fence_after();
      const int ncols = min(a.Nt, a.N - t0);
      const int ot = 2 * x.ot + int(rank);  // this CTA's 128-row weight tile
      const uint32_t tl = tmem_base + uint32_t(buf) * a.acc_cols + (uint32_t(32 * q) << 16);
      for (int c0 = 0; c0 < ncols; c0 += 32) {
        float v[32];
        tmem_ld_32cols(tl + uint32_t(c0), v);
        tmem_wait_ld();
        const int nc = min(32, ncols - c0);
        if (a.splits > 1) {
          // a K range of a split GEMM: the raw f32 partial
          const int o = ot * kBM + 32 * q + lane;
          if (o < a.O) {
            float* pp = a.part + (size_t(x.sp) * a.N + t0 + c0) * a.O + o;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < nc) pp[size_t(i) * a.O] = v[i];
          }
        } else if (EPI == kProjSwiGLU) {
          // lanes 0..63 hold the gate features, lanes 64..127 the matching up
          // features: each half hands the other its values of 16 of the 32
          // columns (column-major exchange, one 128-word row per column), then
          // every warp forms SiLU(gate) * up for its 16 columns - the gate half
          // columns 0..15, the up half 16..31
          const bool gate = q < 2;
          // the columns this thread hands over: 16..31 (gate half) or 0..15
#pragma unroll
          for (int j = 0; j < 16; ++j) upx[j * 128 + 32 * q + lane] = gate ? v[16 + j] : v[j];
          named_bar_sync(1, 128);
          const int f = ot * 64 + 32 * (q & 1) + lane;  // output feature
          const int cb = gate ? 0 : 16;                 // the columns this thread forms
          if (f < a.O / 2) {
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              if (cb + j < nc) {
                const float other = upx[j * 128 + 32 * (q ^ 2) + lane];
                const float g = gate ? v[j] : other;
                const float up = gate ? other : v[16 + j];
                // SiLU(g) up = g up / (1 + e^-g), the quotient by the fast
                // reciprocal (the result is rounded to bf16)
                const float y = __fdividef(g * up, 1.f + __expf(-g));
                a.out[size_t(t0 + c0 + cb + j) * a.ldo + f] = __float2bfloat16_rn(y);
              }
            }
          }
          named_bar_sync(1, 128);
        } else if (EPI == kProjStore && a.vec && ot * kBM + 32 * q + 32 <= a.O) {
          // this warp's 32 features x 32 rows through its 2 KB of the exchange
          // buffer (unused by this epilogue), then 16-byte pieces of each row
          __nv_bfloat16* stg = reinterpret_cast<__nv_bfloat16*>(upx) + q * 1024;
#pragma unroll
          for (int i = 0; i < 32; ++i) stg[i * 32 + lane] = __float2bfloat16_rn(v[i]);
          __syncwarp();
          const int f0 = ot * kBM + 32 * q;  // the warp's first output feature
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int e = lane + 32 * k, row = e >> 2, pc = e & 3;
            if (row < nc)
              *reinterpret_cast<uint4*>(a.out + size_t(t0 + c0 + row) * a.ldo + f0 + 8 * pc) =
                  *reinterpret_cast<const uint4*>(stg + row * 32 + 8 * pc);
          }
          __syncwarp();
        } else {
          const int o = ot * kBM + 32 * q + lane;  // output feature
          if (o < a.O) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              if (i < nc) {
                const size_t at = size_t(t0 + c0 + i) * a.ldo + o;
                float y = v[i];
                if (EPI == kProjResid) y += __bfloat162float(a.res[at]);
                a.out[at] = __float2bfloat16_rn(y);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank != 0)
          mbar_arrive_cluster(tempty_even + uint32_t(buf) * 8u);
        else
          mbar_arrive(tempty + buf);
      }
    }
    if (*epi_abort) flag(a.status, JET_ERR_TIMEOUT);
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA leaves (or frees its TMEM) while the partner's MMAs or
  // copies may still use its shared memory or TMEM
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, a.tmem_cols);
  }
}

// the epilogue of a split GEMM: sum the f32 partials, then store / add the
// residual / SiLU(gate) * up; one thread per output element
template <int EPI>
__global__ void proj_reduce_kernel(const float* __restrict__ part, int splits, int N, int O,
                                   __nv_bfloat16* __restrict__ out, int ldo,
                                   const __nv_bfloat16* res) {
  pdl_begin();
  const int width = EPI == kProjSwiGLU ? O / 2 : O;
  const long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (e >= (long long)N * width) return;
  const int n = int(e / width), c = int(e % width);
  if (EPI == kProjSwiGLU) {
    const int gr = 128 * (c / 64) + c % 64;  // the gate row of feature c; its up row is 64 on
    float g = 0.f, up = 0.f;
    for (int s = 0; s < splits; ++s) {
      const float* row = part + (size_t(s) * N + n) * O;
      g += row[gr];
      up += row[gr + 64];
    }
    out[size_t(n) * ldo + c] = __float2bfloat16_rn(__fdividef(g * up, 1.f + __expf(-g)));
  } else {
    float acc = 0.f;
    for (int s = 0; s < splits; ++s) acc += part[(size_t(s) * N + n) * O + c];
    if (EPI == kProjResid) acc += __bfloat162float(res[size_t(n) * ldo + c]);
    out[size_t(n) * ldo + c] = __float2bfloat16_rn(acc);
  }
}

// A split residual GEMM's epilogue together with the RMSNorm that follows it
// in a decoder layer: one 512-thread block per row (a row's partials need many
// loads in flight; with 128 threads the pass was slower than the two it
// replaces), x = res + the sum of the partials (one rounding), then
// h = x / sqrt(mean(x^2) + eps) * g from the rounded row, in the order of the
// stand-alone RMSNorm kernel (the same results as the two passes). D % 8 == 0;
// res may be out.
constexpr int kNormThreads = 512;
__global__ void __launch_bounds__(kNormThreads)
proj_reduce_norm_kernel(const float* __restrict__ part, int splits, int N, int D,
                        __nv_bfloat16* out, const __nv_bfloat16* res,
                        const __nv_bfloat16* __restrict__ g, float eps,
                        __nv_bfloat16* __restrict__ h) {
  pdl_begin();
  __shared__ float wsum[kNormThreads / 32];
  const int n = blockIdx.x, tid = threadIdx.x;
  if (n >= N) return;
  __nv_bfloat16* xr = out + size_t(n) * D;
  const __nv_bfloat16* rr = res + size_t(n) * D;
  float ss = 0.f;
#pragma unroll 2
  for (int k = tid * 8; k < D; k += kNormThreads * 8) {
    float acc[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i] = 0.f;
    // several splits' loads in flight at once: a block per row has few threads
#pragma unroll 4
    for (int s = 0; s < splits; ++s) {
      const float4* pp = reinterpret_cast<const float4*>(part + (size_t(s) * N + n) * D + k);
      const float4 a0 = pp[0], a1 = pp[1];
      acc[0] += a0.x; acc[1] += a0.y; acc[2] += a0.z; acc[3] += a0.w;
      acc[4] += a1.x; acc[5] += a1.y; acc[6] += a1.z; acc[7] += a1.w;
    }
    const uint4 rv = *reinterpret_cast<const uint4*>(rr + k);
    const __nv_bfloat162* pr = reinterpret_cast<const __nv_bfloat162*>(&rv);
    uint4 xv;
    __nv_bfloat162* px = reinterpret_cast<__nv_bfloat162*>(&xv);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(pr[i]);
      px[i] = __floats2bfloat162_rn(acc[2 * i] + f.x, acc[2 * i + 1] + f.y);
    }
    *reinterpret_cast<uint4*>(xr + k) = xv;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(px[i]);
      ss = fmaf(f.x, f.x, fmaf(f.y, f.y, ss));
    }
  }
  ss = warp_sum(ss);
  if ((tid & 31) == 0) wsum[tid >> 5] = ss;
  __syncthreads();
  ss = 0.f;
#pragma unroll
  for (int w = 0; w < kNormThreads / 32; ++w) ss += wsum[w];
  const float inv = 1.f / sqrtf(ss / float(D) + eps);
  __nv_bfloat16* hr = h + size_t(n) * D;
  for (int k = tid * 8; k < D; k += kNormThreads * 8) {
    const uint4 v = *reinterpret_cast<const uint4*>(xr + k);  // this thread's own writes
    const uint4 gv = *reinterpret_cast<const uint4*>(g + k);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&v);
    const __nv_bfloat162* pg = reinterpret_cast<const __nv_bfloat162*>(&gv);
    uint4 o4;
    __nv_bfloat162* po = reinterpret_cast<__nv_bfloat162*>(&o4);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __bfloat1622float2(p[i]), gg = __bfloat1622float2(pg[i]);
      po[i] = __floats2bfloat162_rn(f.x * inv * gg.x, f.y * inv * gg.y);
    }
    *reinterpret_cast<uint4*>(hr + k) = o4;
  }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// row-major bf16 [rows, K] with row stride ld elements; box 64 x box_rows,
// 128-byte swizzle
bool encode_rows(CUtensorMap* map, const void* base, int rows, int K, int ld, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cuuint64_t(K), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(ld) * 2};
  const cuuint32_t box[2] = {cuuint32_t(kBK), cuuint32_t(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

// clusters of two CTAs of `kern` that can be resident at once (one CTA per SM:
// the SM pairs the GPCs offer); asked once per kernel
template <typename K>
int max_pairs(K kern, size_t smem) {
  static int cached = 0;
  if (cached > 0) return cached;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute cl{};
  cl.id = cudaLaunchAttributeClusterDimension;
  cl.val.clusterDim.x = 2;
  cl.val.clusterDim.y = 1;
  cl.val.clusterDim.z = 1;
  cfg.attrs = &cl;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n < 1)
    n = std::max(1, sm_count() / 2);
  cached = n;
  return n;
}

// the RMSNorm a residual projection's output feeds (h null: none)
struct Norm {
  const void* g;
  float eps;
  void* h;
};

template <int EPI>
cudaError_t launch_reduce(const ProjArgs& a, float* part, int N, int O, void* out, int ldo,
                          const void* res, cudaStream_t st);

struct Tiling {
  int n_tt, Nt, otiles, groups, nkb, splits;  // groups: 256-row weight slices
};

// token tiles of at most 256 rows (a multiple of 16: each CTA of a pair holds
// half); units of 256 weight rows on CTA pairs; K split while the units still
// fit the 76 SM pairs once, keeping at least 8 K slices per unit. A function
// of the shapes only, so that the workspace planned for a call matches the
// launch.
constexpr int kPlanSMs = 152;
Tiling tiling(int N, int O, int K, bool split) {
  Tiling t{};
  t.n_tt = (N + kMaxNt - 1) / kMaxNt;
  t.Nt = ((N + t.n_tt - 1) / t.n_tt + 15) / 16 * 16;
  t.n_tt = (N + t.Nt - 1) / t.Nt;
  t.otiles = (O + kBM - 1) / kBM;
  t.groups = (t.otiles + 1) / 2;
  t.nkb = (K + kBK - 1) / kBK;
  const int units = t.groups * t.n_tt;
  t.splits = 1;
  while (split && units * (t.splits + 1) <= kPlanSMs / 2 && t.nkb / (t.splits + 1) >= 8)
    ++t.splits;
  return t;
}

template <int EPI>
cudaError_t launch_epi(const void* x, int N, int K, int ldx, const void* w, int O, void* out,
                       int ldo, const void* res, float* part, int* status, cudaStream_t st,
                       const Norm& nm, int* splits_out = nullptr) {
  const Tiling tl = tiling(N, O, K, part != nullptr);
  const int n_tt = tl.n_tt, Nt = tl.Nt;
  ProjArgs a{};
  a.wait_ns = wait_budget_ns();
  a.hold_first = test_stall();
  a.part = part;
  a.splits = part ? tl.splits : 1;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.res = static_cast<const __nv_bfloat16*>(res);
  a.status = status;
  a.N = N;
  a.O = O;
  a.K = K;
  a.ldo = ldo;
  a.vec = (ldo % 8 == 0) && (reinterpret_cast<uintptr_t>(out) % 16 == 0);
  a.Nt = Nt;
  a.n_tt = n_tt;
  a.units = tl.groups * n_tt * a.splits;
  a.nkb = (K + kBK - 1) / kBK;
  a.acc_cols = Nt <= 128 ? 128 : 256;
  a.tmem_cols = 2 * a.acc_cols;
  const int b_rows = Nt / 2;  // token-tile rows one CTA loads
  const int stage_bytes = kBM * 128 + b_rows * 128;
  a.stages = std::min(8, (kSmemLimit - 1024 - kFixedSmem) / stage_bytes);
  const size_t smem = 1024 + size_t(a.stages) * stage_bytes + kFixedSmem;
  CUtensorMap tmW, tmX;
  if (!encode_rows(&tmW, w, O, K, K, kBM) || !encode_rows(&tmX, x, N, K, ldx, b_rows))
    return cudaErrorInvalidValue;
  auto kern = proj_tc_kernel<EPI>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  const int clusters = std::max(1, std::min(a.units, max_pairs(kern, smem)));
  e = launch_pdl_pairs(kern, dim3(unsigned(2 * clusters)), dim3(kThreads), smem, st, tmW, tmX, a);
  if (e != cudaSuccess) return e;
  if (splits_out) {
    // the caller reduces the partials itself
    *splits_out = a.splits;
    if (a.splits > 1) return cudaSuccess;
  }
  const bool norm = EPI == kProjResid && nm.h != nullptr;
  if (norm && a.splits > 1 && ldo == O && O % 8 == 0)
    return launch_pdl(proj_reduce_norm_kernel, dim3(unsigned(N)), dim3(kNormThreads), 0, st,
                      static_cast<const float*>(part), a.splits, N, O,
                      static_cast<__nv_bfloat16*>(out), static_cast<const __nv_bfloat16*>(res),
                      static_cast<const __nv_bfloat16*>(nm.g), nm.eps,
                      static_cast<__nv_bfloat16*>(nm.h));
  if (a.splits > 1) {
    e = launch_reduce<EPI>(a, part, N, O, out, ldo, res, st);
    if (e != cudaSuccess) return e;
  }
  return norm ? launch_rmsnorm(out, nm.g, N, O, nm.eps, nm.h, st) : cudaSuccess;
}

template <int EPI>
cudaError_t launch_reduce(const ProjArgs& a, float* part, int N, int O, void* out, int ldo,
                          const void* res, cudaStream_t st) {
  const long long total = (long long)N * (EPI == kProjSwiGLU ? O / 2 : O);
  return launch_pdl(proj_reduce_kernel<EPI>, dim3(unsigned((total + 255) / 256)), dim3(256), 0, st,
                    static_cast<const float*>(part), a.splits, N, O,
                    static_cast<__nv_bfloat16*>(out), ldo,
                    static_cast<const __nv_bfloat16*>(res));
}

}  // namespace

cudaError_t launch_proj_gates(const jet_layout& lay, const void* x, int K, const void* w, int O,
                              void* z, int Hl, int dv, void* lq_all, void* lq, void* lk, void* lv,
                              float* alpha, float* beta, float* part, int* status,
                              cudaStream_t st) {
  const int N = lay.n.N;
  if (N <= 0 || O <= 0) return cudaSuccess;
  int splits = 1;
  cudaError_t e = launch_epi<kProjStore>(x, N, K, K, w, O, z, O, nullptr, part, status, st,
                                         Norm{nullptr, 0.f, nullptr}, &splits);
  if (e != cudaSuccess) return e;
  if (splits > 1)
    return launch_reduce_gates(lay, part, splits, Hl, dv, lq_all, lq, lk, lv, alpha, beta, status,
                               st);
  return launch_gates(lay, z, Hl, dv, lq_all, lq, lk, lv, alpha, beta, status, st);
}

cudaError_t launch_proj_qkv(const jet_layout& lay, const void* x, int K, const void* w, int qw,
                            int kw, void* z, void* q, void* kc, void* vc, float* part,
                            int* status, cudaStream_t st) {
  const int N = lay.n.N, O = qw + 2 * kw;
  if (N <= 0 || O <= 0) return cudaSuccess;
  int splits = 1;
  cudaError_t e = launch_epi<kProjStore>(x, N, K, K, w, O, z, O, nullptr, part, status, st,
                                         Norm{nullptr, 0.f, nullptr}, &splits);
  if (e != cudaSuccess) return e;
  if (splits > 1) return launch_reduce_qkv(lay, part, splits, qw, kw, q, kc, vc, status, st);
  return launch_split_qkv(lay, z, qw, kw, q, kc, vc, status, st);
}

size_t proj_partial_bytes(int N, int O, int K) {
  const Tiling t = tiling(N, O, K, true);
  return t.splits > 1 ? size_t(t.splits) * N * O * sizeof(float) : 0;
}

cudaError_t launch_proj(int epi, const void* x, int N, int K, int ldx, const void* w, int O,
                        void* out, int ldo, const void* res, float* part, int* status,
                        cudaStream_t st, const void* norm_g, float norm_eps, void* norm_h) {
  if (N <= 0 || O <= 0) return cudaSuccess;
  const Norm nm{norm_g, norm_eps, norm_h};
  if (epi == kProjResid)
    return launch_epi<kProjResid>(x, N, K, ldx, w, O, out, ldo, res, part, status, st, nm);
  if (epi == kProjSwiGLU)
    return launch_epi<kProjSwiGLU>(x, N, K, ldx, w, O, out, ldo, res, part, status, st, nm);
  return launch_epi<kProjStore>(x, N, K, ldx, w, O, out, ldo, res, part, status, st, nm);
}

}  // namespace jet
