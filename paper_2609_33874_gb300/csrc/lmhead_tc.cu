// LM head on the 5th-generation tensor cores with an on-chip log-sum-exp
// epilogue and target gather (Eq. 1, Eq. 2; Sec. 4.2: logits never leave the
// chip, only the needed log-probabilities do).
//
// Orientation: the vocabulary is the MMA's M dimension (128 rows of w_lm per
// tile = the 128 TMEM lanes) and the query rows are its N dimension (a token
// tile of up to 256 rows). Candidate-scoring batches have a few hundred rows
// at most per tile, so this keeps the tensor-core work equal to the useful
// work instead of padding the rows to 128-row multiples; the weights stream
// through once per token tile.
//
// Pipeline (one persistent CTA per SM, 6 warps):
//   warp 0      TMA producer: 128x64 w_lm tile + Nt x 64 hidden tile per stage,
//               both 128-byte swizzled, into a ring of shared-memory stages
//   warp 1      TMEM allocator and MMA issuer: 4 x tcgen05.mma (K = 16) per
//               stage into one of two TMEM accumulators (double buffered)
//   warps 2..5  epilogue: each warp reads its 32 TMEM lanes (32 vocabulary
//               entries) x 32 token columns at a time, reduces (max, sum of
//               2^x) per token across its lanes with a butterfly exchange,
//               combines the 4 warps through shared memory and writes one
//               partial per (token, vocabulary tile); target logits are read
//               straight from TMEM.
// Partials use base 2: m = max z log2(e), s = sum 2^(z log2(e) - m).
//
// The e4m3 instantiation (low-precision LM head; Appendix A: the paper's
// models run with 8-bit and 4-bit weights) keeps the same byte geometry - a
// 128-byte K slice is 128 e4m3 elements - issues tcgen05.mma kind::f8f6f4
// (K = 32 per instruction) and applies the per-row weight scale and per-token
// hidden scale to each logit in the epilogue: z = s_w[v] s_h[n] acc.
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

constexpr int kBM = kVocabTile;     // 128 vocabulary rows per tile (MMA M, TMEM lanes)
constexpr int kBK = 64;             // bf16 hidden elements per stage: 128 bytes
constexpr int kBKBytes = 128;       // bytes of one K slice of a row, either element type
constexpr int kThreads = 192;
constexpr int kMaxNt = 256;
constexpr uint64_t kWaitNs = 2000000000ull;  // budget of one wait
constexpr uint64_t kDrainNs = 200000000ull;  // budget of the drain after an abort
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kNegBig = -1.0e30f;          // logit of a vocabulary row beyond V
constexpr int kSmemLimit = 232448;           // opt-in shared memory per block
constexpr int kFixedSmem = 4 * kMaxNt * 8 + 128 * 16 + 64 * 8 + 64 + kMaxNt * 4;

struct TcArgs {
  const int32_t* target_ids;
  const int32_t* tgt_row;
  const int32_t* row_tgt_offset;
  const int32_t* row_tgt_index;
  float2* part;
  float* z_tgt;
  const float* w_scale;  // e4m3: [V] per vocabulary row
  const float* h_scale;  // e4m3: [N] per token
  int* status;
  int N, T, V, D;
  int Nt, n_tt, units, nkb, stages, vtiles;
  uint32_t tmem_cols;
};

__device__ __forceinline__ void combine(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  const float e = ex2(fminf(m, m2) - M);
  s = (m >= m2) ? fmaf(s2, e, s) : fmaf(s, e, s2);
  m = M;
}

// One butterfly stage: lanes exchange the half of their columns they do not
// keep with the partner lane `o` away and combine the kept half.
template <int O>
__device__ __forceinline__ void butterfly(float* m, float* s, int lane) {
  const bool up = (lane & O) != 0;
#pragma unroll
  for (int i = 0; i < O; ++i) {
    const float km = up ? m[i + O] : m[i], ks = up ? s[i + O] : s[i];
    const float sm = up ? m[i] : m[i + O], ss = up ? s[i] : s[i + O];
    const float rm = __shfl_xor_sync(0xffffffffu, sm, O);
    const float rs = __shfl_xor_sync(0xffffffffu, ss, O);
    float M = km, S = ks;
    combine(M, S, rm, rs);
    m[i] = M;
    s[i] = S;
  }
}

// D (+)= A B^T, A and B e4m3 codes described in shared memory (K = 32)
__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Instruction descriptor of kind::f8f6f4: A and B e4m3 (format 0, K-major),
// f32 accumulator, shape M x N.
constexpr uint32_t idesc_e4m3_f32(int M, int N) {
  return (1u << 4) | (uint32_t(N >> 3) << 17) | (uint32_t(M >> 4) << 24);
}

template <bool F8>
__global__ void __launch_bounds__(kThreads, 1)
lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmH,
                 const TcArgs a) {
  constexpr int kBKe = F8 ? kBKBytes : kBK;  // elements of one K slice
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t a_bytes = kBM * 128, b_bytes = uint32_t(a.Nt) * 128;
  const uint32_t stage_bytes = a_bytes + b_bytes;
  float2* red = reinterpret_cast<float2*>(smem + size_t(a.stages) * stage_bytes);  // [4][256]
  int4* hits = reinterpret_cast<int4*>(red + 4 * kMaxNt);                          // [128]
  float* hs = reinterpret_cast<float*>(hits + 128);                                // [256]
  uint64_t* full = reinterpret_cast<uint64_t*>(hs + kMaxNt);
  uint64_t* empty = full + a.stages;
  uint64_t* tfull = empty + a.stages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  int* hit_count = reinterpret_cast<int*>(tmem_slot + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(hit_count + 1);
  volatile int* epi_abort = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull + b, 1);
      mbar_init(tempty + b, 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    *epi_abort = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmH);
  }
  // global memory and TMEM only after the previous kernel of the stream is done
  pdl_begin();
  if (warp == 1) {
    tmem_alloc(tmem_slot, a.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t buf_cols = a.tmem_cols / 2;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_h = policy_evict_last();
      int s = 0;
      uint32_t ph = 0, issued = 0, issued_par = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
        const int v0 = (u / a.n_tt) * kBM, t0 = (u % a.n_tt) * a.Nt;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1u, kWaitNs, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + size_t(s) * stage_bytes;
          mbar_arrive_expect_tx(full + s, stage_bytes);
          tma_load_2d(sa, &tmW, full + s, kb * kBKe, v0, pol_w);
          tma_load_2d(sa + a_bytes, &tmH, full + s, kb * kBKe, t0, pol_h);
          issued |= 1u << s;
          issued_par = (issued_par & ~(1u << s)) | (ph << s);
          if (++s == a.stages) {
            s = 0;
            ph ^= 1u;
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        // let every copy already issued land before the CTA can exit
        for (int t = 0; t < a.stages; ++t)
          if (issued & (1u << t)) mbar_wait(full + t, (issued_par >> t) & 1u, kDrainNs, nullptr);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = F8 ? idesc_e4m3_f32(kBM, a.Nt) : idesc_bf16_f32(kBM, a.Nt);
      int s = 0, local = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x, ++local) {
        const int buf = local & 1;
        const uint32_t tph = (local >> 1) & 1;
        if (!mbar_wait(tempty + buf, tph ^ 1u, kWaitNs, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + buf * buf_cols;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(full + s, ph, kWaitNs, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + size_t(s) * stage_bytes), sb = sa + a_bytes;
          // 32 bytes of K per instruction: 16 bf16 or 32 e4m3 elements
#pragma unroll
          for (int k = 0; k < kBKBytes / 32; ++k) {
            if (F8)
              mma_e4m3(d_tmem, desc_k_sw128(sa + 32 * k), desc_k_sw128(sb + 32 * k), idesc,
                       (kb | k) != 0);
            else
              mma_f16(d_tmem, desc_k_sw128(sa + 32 * k), desc_k_sw128(sb + 32 * k), idesc,
                      (kb | k) != 0);
          }
          mma_commit(empty + s);  // frees the stage once these MMAs have read it
          if (++s == a.stages) {
            s = 0;
            ph ^= 1u;
          }
        }
        if (!ok) break;
        mma_commit(tfull + buf);  // accumulator complete
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        mma_commit(drain);
        mbar_wait(drain, 0, kDrainNs, nullptr);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;          // TMEM lane quadrant this warp may access
    const int et = threadIdx.x - 64;  // 0..127
    const int vrow = q * 32 + lane;   // vocabulary row within the tile
    int local = 0;
    for (int u = blockIdx.x; u < a.units; u += gridDim.x, ++local) {
      const int buf = local & 1;
      const uint32_t tph = (local >> 1) & 1;
      const int vt = u / a.n_tt;
      const int v0 = vt * kBM, t0 = (u % a.n_tt) * a.Nt;
      const bool ok = warp_mbar_wait(tfull + buf, tph, kWaitNs, abort_flag);
      if (!ok || *abort_flag) *epi_abort = 1;
      named_bar_sync(1, 128);
      if (*epi_abort) break;
      tc_fence_after();
      const uint32_t tcol = tmem_base + buf * buf_cols;
      const uint32_t tl = tcol + (uint32_t(32 * q) << 16);
      const int ncols = min(a.Nt, a.N - t0);
      const bool row_valid = v0 + vrow < a.V;
      // e4m3: this row's weight scale, and the unit's token scales in shared memory
      float wsc = 1.f;
      if (F8) {
        wsc = row_valid ? a.w_scale[v0 + vrow] : 0.f;
        for (int c = et; c < ncols; c += 128) hs[c] = a.h_scale[t0 + c];
        named_bar_sync(1, 128);
      }

      // target gather: rows [t0, t0 + ncols) whose target lies in this tile
      const int j_begin = a.row_tgt_offset[t0], j_end = a.row_tgt_offset[t0 + ncols];
      for (int base = j_begin; base < j_end; base += 128) {
        if (et == 0) *hit_count = 0;
        named_bar_sync(1, 128);
        const int jj = base + et;
        if (jj < j_end) {
          const int j = a.row_tgt_index[jj];
          if (j >= 0 && j < a.T) {
            const int off = a.target_ids[j] - v0;
            const int col = a.tgt_row[j] - t0;
            if (off >= 0 && off < kBM && col >= 0 && col < ncols) {
              const int h = atomicAdd(hit_count, 1);
              hits[h] = make_int4(j, off >> 5, off & 31, col);
            }
          } else {
            flag(a.status, JET_ERR_DEVICE);
          }
        }
        named_bar_sync(1, 128);
        const int nh = *hit_count;
        for (int h = 0; h < nh; ++h) {
          const int4 hv = hits[h];
          if (hv.y == q) {
            const float z = tmem_ld_1col(tl + uint32_t(hv.w));
            tmem_wait_ld();
            if (lane == hv.z) a.z_tgt[hv.x] = F8 ? z * wsc * hs[hv.w] : z;
          }
        }
        named_bar_sync(1, 128);
      }

      // (max, sum 2^x) per token column over this warp's 32 vocabulary rows
      for (int c0 = 0; c0 < ncols; c0 += 32) {
        float v[32];
        tmem_ld_32cols(tl + uint32_t(c0), v);
        tmem_wait_ld();
        if (F8) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] *= wsc * hs[c0 + i];
        }
        float m[16], s[16];
        {
          const bool up = (lane & 16) != 0;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float a0 = row_valid ? v[i] * kLog2e : kNegBig;
            const float a1 = row_valid ? v[i + 16] * kLog2e : kNegBig;
            const float keep = up ? a1 : a0, send = up ? a0 : a1;
            const float recv = __shfl_xor_sync(0xffffffffu, send, 16);
            const float M = fmaxf(keep, recv);
            m[i] = M;
            s[i] = 1.f + ex2(fminf(keep, recv) - M);
          }
        }
        butterfly<8>(m, s, lane);
        butterfly<4>(m, s, lane);
        butterfly<2>(m, s, lane);
        butterfly<1>(m, s, lane);
        red[q * kMaxNt + c0 + lane] = make_float2(m[0], s[0]);
      }
      // the accumulator can be overwritten now
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty + buf);
      named_bar_sync(1, 128);
      for (int c = et; c < ncols; c += 128) {
        float M = red[c].x, S = red[c].y;
#pragma unroll
        for (int w = 1; w < 4; ++w) combine(M, S, red[w * kMaxNt + c].x, red[w * kMaxNt + c].y);
        a.part[size_t(t0 + c) * a.vtiles + vt] = make_float2(M, S);
      }
      named_bar_sync(1, 128);
    }
    if (*epi_abort) flag(a.status, JET_ERR_TIMEOUT);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, a.tmem_cols);
  }
}

// ---- host side --------------------------------------------------------------
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

// row-major [rows, D] matrix of bf16 (esize 2) or e4m3 codes (esize 1), box of
// one 128-byte K slice x box_rows rows, 128-byte swizzle
bool encode_kmajor(CUtensorMap* map, const void* base, int rows, int D, int box_rows, int esize) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cuuint64_t(D), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(D) * esize};
  const cuuint32_t box[2] = {cuuint32_t(kBKBytes / esize), cuuint32_t(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, esize == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, 2,
            const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

}  // namespace

namespace {

// one launch of the LM head on bf16 operands (F8 false) or e4m3 codes with
// per-row weight scales and per-token hidden scales (F8 true)
template <bool F8>
cudaError_t launch_head(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                        const void* hidden, const float* h_scale, const void* w_lm,
                        const float* w_scale, void* ws, int* status, cudaStream_t st) {
  const jet_sizes& n = lay.n;
  int n_tt = (n.N + kMaxNt - 1) / kMaxNt;
  const int Nt = ((n.N + n_tt - 1) / n_tt + 15) / 16 * 16;
  n_tt = (n.N + Nt - 1) / Nt;
  const int esize = F8 ? 1 : 2;
  TcArgs a{};
  a.target_ids = lay.target_ids;
  a.tgt_row = lay.tgt_row;
  a.row_tgt_offset = lay.row_tgt_offset;
  a.row_tgt_index = lay.row_tgt_index;
  char* base = static_cast<char*>(ws);
  a.part = reinterpret_cast<float2*>(base + plan.part_off);
  a.z_tgt = reinterpret_cast<float*>(base + plan.ztgt_off);
  a.w_scale = w_scale;
  a.h_scale = h_scale;
  a.status = status;
  a.N = n.N;
  a.T = n.T;
  a.V = n.V;
  a.D = d.D;
  a.Nt = Nt;
  a.n_tt = n_tt;
  a.units = plan.vtiles * n_tt;
  a.vtiles = plan.vtiles;
  a.nkb = (d.D * esize + kBKBytes - 1) / kBKBytes;
  a.tmem_cols = Nt <= 128 ? 256 : 512;
  const int stage_bytes = kBM * kBKBytes + Nt * kBKBytes;
  a.stages = std::min(8, (kSmemLimit - 1024 - kFixedSmem) / stage_bytes);
  const size_t smem = 1024 + size_t(a.stages) * stage_bytes + kFixedSmem;

  CUtensorMap tmW, tmH;
  if (!encode_kmajor(&tmW, w_lm, n.V, d.D, kBM, esize) ||
      !encode_kmajor(&tmH, hidden, n.N, d.D, Nt, esize))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(lmhead_tc_kernel<F8>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  int sms = sm_count();
  if (d.max_sms > 0) sms = std::min(sms, d.max_sms);
  const int grid = std::max(1, std::min(a.units, sms));
  return launch_pdl(lmhead_tc_kernel<F8>, dim3(grid), dim3(kThreads), smem, st, tmW, tmH, a);
}

}  // namespace

cudaError_t launch_lmhead_tc(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const void* hidden, const void* w_lm, void* ws, int* status,
                             cudaStream_t st) {
  return launch_head<false>(lay, d, plan, hidden, nullptr, w_lm, nullptr, ws, status, st);
}

cudaError_t launch_lmhead_e4m3(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                               const uint8_t* h_q, const float* h_scale, const uint8_t* w_q,
                               const float* w_scale, void* ws, int* status, cudaStream_t st) {
  return launch_head<true>(lay, d, plan, h_q, h_scale, w_q, w_scale, ws, status, st);
}

}  // namespace jet
