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
//
// The w4 instantiation (4-bit weights: E2M1 codes with a power-of-two exponent
// per 32-element block under a float32 row scale) streams the weights at half
// the e4m3 bytes and multiplies them on the block-scaled tensor-core path:
// the TMA unpacks a 128 x 128 tile of packed codes into the padded layout
// tcgen05.mma kind::mxf8f6f4 reads for E2M1 operands (16 codes in the low 8
// bytes of each 16-byte chunk, 128-byte swizzled like an e4m3 tile), a bulk
// copy brings the tile's 512-byte chunk of UE8M0 block scale factors, and the
// MMA thread moves the chunk into TMEM (tcgen05.cp, 32 x 128 bits replicated
// to the four lane quadrants: row 32 j + i of the tile at lane 32 j + i,
// column j, byte = block) before the four block-scaled MMAs of the slice.
// The hidden states' scale factors are all 1 (their float32 per-token scale
// is applied in the epilogue, as in the e4m3 instantiation); the hardware
// reads them at lane n % 32, column n / 32, so eight columns of 0x7F cover
// any token tile. Each product 2^e value(code) x code(h) is exact and
// accumulated in float32, so the arithmetic is the same as widening the codes
// to e4m3, without any widening work on the SMs.
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
enum { kFmtBf16 = 0, kFmtE4m3 = 1, kFmtW4 = 2, kFmtMx8 = 3 };
constexpr int kMaxNt = 256;
// block-scaled formats: token tiles of at most 224 columns leave room in TMEM
// (512 columns) for the two accumulators and the scale-factor slots
constexpr int kMaxNtBs = 224;
constexpr int kSfbCols = 8;
constexpr int kSfaSlot = 8;   // TMEM columns per stage's weight scale factors (4 used)
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
  const uint8_t* w_sf;   // w4, mxfp8: the weights' scale factors, a 512-byte chunk per tile
  const uint8_t* h_sf;   // mxfp8: the hidden states' scale factors, two chunks per tile
  int* status;
  int N, T, V, D;
  int Nt, n_tt, units, nkb, stages, vtiles;
  uint32_t tmem_cols;
  uint32_t buf_cols;     // columns of one accumulator
  uint32_t sfb_col;      // the hidden side's scale factors: w4 one slot (all 1),
                         // mxfp8 kSfaSlot columns per stage
  uint32_t sfa_col;      // the weight scale factors, kSfaSlot columns per stage
  uint64_t wait_ns;  // budget of one bounded wait (jet_set_wait_budget_ns)
  int hold_first;    // test hook (jet_set_test_stall): withhold the first stage's loads
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

// D (+)= (A x sf_A) (B x sf_B)^T with A E2M1 codes and B e4m3 codes in shared
// memory, one UE8M0 scale factor per 32-element block of K in TMEM (K = 32:
// the instruction descriptor's scale-factor ids pick the byte)
__device__ __forceinline__ void mma_mx(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                       uint32_t idesc, uint32_t sfa_tmem, uint32_t sfb_tmem,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %6, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X "
      "[%0], %1, %2, %3, [%4], [%5], p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(sfa_tmem), "r"(sfb_tmem), "r"(accumulate)
      : "memory");
}

// Instruction descriptor of kind::mxf8f6f4 with block scaling: A of format
// `afmt` (E2M1 = 5, e4m3 = 0), B e4m3 (format 0), both K-major, UE8M0 scale
// factors, shape M x N; block `k` of the 4 in a scale-factor word for both
// operands.
__host__ __device__ constexpr uint32_t idesc_mx(uint32_t afmt, int M, int N, int k) {
  return (uint32_t(k) << 4) | (afmt << 7) | (0u << 10) | (uint32_t(N >> 3) << 17) | (1u << 23) |
         (uint32_t(M >> 4) << 24) | (uint32_t(k) << 29);
}

// A 32 x 16-byte matrix in shared memory (rows 16 bytes apart) into TMEM,
// replicated to all four 32-lane quadrants: row i at lane 32 q + i, its four
// 32-bit words in columns taddr .. taddr + 3.
__device__ __forceinline__ void tmem_cp_32x128(uint32_t taddr, uint32_t smem_addr) {
  uint64_t d = 0;
  d |= uint64_t((smem_addr >> 4) & 0x3FFFu);  // start address
  d |= uint64_t(1) << 16;                     // leading byte offset (one 16-byte column)
  d |= uint64_t(128 >> 4) << 32;              // stride byte offset: 8 rows x 16 bytes
  d |= uint64_t(1) << 46;                     // descriptor version (sm_100 family)
  asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(d)
               : "memory");
}

// untiled bulk copy global -> shared memory, completing `bytes` on `bar`
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tmem_st_8cols(uint32_t taddr, uint32_t v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %1, %1, %1, %1, %1, %1, %1};" ::"r"(taddr),
      "r"(v)
      : "memory");
}

template <int FMT>
__global__ void __launch_bounds__(kThreads, 1)
lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmH,
                 const TcArgs a) {
  constexpr bool F8 = FMT != kFmtBf16;   // 8-bit hidden codes in the MMA
  constexpr bool W4 = FMT == kFmtW4;     // 4-bit weights, block-scaled MMA
  constexpr bool MX = FMT == kFmtMx8;    // e4m3 blocks on both sides, block-scaled MMA
  constexpr bool ROWSC = FMT == kFmtE4m3 || W4;  // float32 scales per weight row and token
  constexpr int kBKe = F8 ? kBKBytes : kBK;  // elements of one K slice
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t a_bytes = kBM * 128, b_bytes = uint32_t(a.Nt) * 128;
  // a stage holds the weight and hidden tiles of one K slice (w4: the weight
  // tile as the TMA unpacks it, 1 byte per code) and the slice's scale-factor
  // chunks: w4 the weights' 512 bytes (in a 1 KB slot), mxfp8 also the hidden
  // states' two chunks (a 2 KB slot), keeping stages 1 KB aligned
  const uint32_t stage_bytes = a_bytes + b_bytes + (W4 ? 1024u : MX ? 2048u : 0u);
  float2* red = reinterpret_cast<float2*>(smem + size_t(a.stages) * stage_bytes);
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
  const uint32_t buf_cols = a.buf_cols;
  if (W4) {
    // the hidden side's scale factors: 1 (UE8M0 127) in every byte the MMA
    // may read, written once by the epilogue warps (each to its lane quadrant)
    if (warp >= 2) {
      tmem_st_8cols(tmem_base + (uint32_t(32 * (warp & 3)) << 16) + a.sfb_col, 0x7F7F7F7Fu);
      tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
  }

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_h = policy_evict_last();
      // the weight bytes one stage brings: bf16 or e4m3 tile, or packed
      // 4-bit codes (half the unpacked tile) and their scale-factor chunk;
      // mxfp8 adds both operands' chunks
      const uint32_t w_tx = W4 ? a_bytes / 2 + kW4ScaleBytes
                               : MX ? a_bytes + 3 * kW4ScaleBytes : a_bytes;
      int s = 0;
      uint32_t ph = 0, issued = 0, issued_par = 0;
      bool ok = true, hold = a.hold_first != 0;
      for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
        const int vt = u / a.n_tt, v0 = vt * kBM, t0 = (u % a.n_tt) * a.Nt;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1u, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + size_t(s) * stage_bytes;
          if (hold) {
            hold = false;  // test hook: this stage never fills
          } else {
            mbar_arrive_expect_tx(full + s, w_tx + b_bytes);
            tma_load_2d(sa, &tmW, full + s, kb * kBKe, v0, pol_w);
            tma_load_2d(sa + a_bytes, &tmH, full + s, kb * kBKe, t0, pol_h);
            if (W4 || MX)
              bulk_load(sa + a_bytes + b_bytes,
                        a.w_sf + (size_t(vt) * a.nkb + kb) * kW4ScaleBytes, kW4ScaleBytes,
                        full + s, pol_w);
            if (MX)
              bulk_load(sa + a_bytes + b_bytes + kW4ScaleBytes,
                        a.h_sf + (size_t(u % a.n_tt) * a.nkb + kb) * 2 * kW4ScaleBytes,
                        2 * kW4ScaleBytes, full + s, pol_h);
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
        if (!mbar_wait(tempty + buf, tph ^ 1u, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + buf * buf_cols;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(full + s, ph, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + size_t(s) * stage_bytes);
          const uint32_t sb = sa + a_bytes;
          if (W4 || MX) {
            // the slice's weight scale factors into this stage's 4 columns
            // (mxfp8: the hidden states' too, 4 columns per 128 token rows);
            // the MMAs after them in this thread's order read them
            const uint32_t sfa = tmem_base + a.sfa_col + kSfaSlot * s;
            const uint32_t sfb = MX ? tmem_base + a.sfb_col + kSfaSlot * s : tmem_base + a.sfb_col;
            tmem_cp_32x128(sfa, sb + b_bytes);
            if (MX) {
              tmem_cp_32x128(sfb, sb + b_bytes + kW4ScaleBytes);
              if (a.Nt > 128) tmem_cp_32x128(sfb + 4, sb + b_bytes + 2 * kW4ScaleBytes);
            }
#pragma unroll
            for (int k = 0; k < 4; ++k)
              mma_mx(d_tmem, desc_k_sw128(sa + 32 * k), desc_k_sw128(sb + 32 * k),
                     idesc_mx(W4 ? 5u : 0u, kBM, a.Nt, k), sfa, sfb, (kb | k) != 0);
          } else {
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
      const bool ok = warp_mbar_wait(tfull + buf, tph, a.wait_ns, abort_flag);
      if (!ok || *abort_flag) *epi_abort = 1;
      named_bar_sync(1, 128);
      if (*epi_abort) break;
      tc_fence_after();
      const uint32_t tcol = tmem_base + buf * buf_cols;
      const uint32_t tl = tcol + (uint32_t(32 * q) << 16);
      const int ncols = min(a.Nt, a.N - t0);
      const bool row_valid = v0 + vrow < a.V;
      // e4m3, w4: this row's weight scale, and the unit's token scales in
      // shared memory (mxfp8 needs none: its block scales are in the MMA)
      float wsc = 1.f;
      if (ROWSC) {
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
            if (lane == hv.z) a.z_tgt[hv.x] = ROWSC ? z * wsc * hs[hv.w] : z;
          }
        }
        named_bar_sync(1, 128);
      }

      // (max, sum 2^x) per token column over this warp's 32 vocabulary rows
      for (int c0 = 0; c0 < ncols; c0 += 32) {
        float v[32];
        tmem_ld_32cols(tl + uint32_t(c0), v);
        tmem_wait_ld();
        if (ROWSC) {
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

// the 4-bit code region [rows, kd] (kd codes per row, two per byte, element
// 2 j in the low nibble of byte j; kd a multiple of 128): boxes of 128 codes x
// 128 rows, unpacked by the TMA to one byte per code (16 codes in the low 8
// bytes of each 16-byte chunk), 128-byte swizzled
bool encode_w4_codes(CUtensorMap* map, const void* base, int rows, int kd) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {cuuint64_t(kd), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(kd) / 2};
  const cuuint32_t box[2] = {128, cuuint32_t(kBM)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_16U4_ALIGN16B, 2, const_cast<void*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

}  // namespace

namespace {

// one launch of the LM head on bf16 operands, or e4m3 hidden codes with e4m3
// or block-scaled 4-bit weights, per-row weight scales and per-token hidden scales
template <int FMT>
cudaError_t launch_head(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                        const void* hidden, const float* h_scale, const void* w_lm,
                        const float* w_scale, void* ws, int* status, cudaStream_t st,
                        const uint8_t* w_sf = nullptr, const uint8_t* h_sf = nullptr) {
  constexpr bool F8 = FMT != kFmtBf16, W4 = FMT == kFmtW4, MX = FMT == kFmtMx8;
  const jet_sizes& n = lay.n;
  int n_tt = 0, Nt = 0;
  if (W4 || MX) {
    mx_token_tiling(n.N, &Nt, &n_tt);
  } else {
    n_tt = (n.N + kMaxNt - 1) / kMaxNt;
    Nt = ((n.N + n_tt - 1) / n_tt + 15) / 16 * 16;
    n_tt = (n.N + Nt - 1) / Nt;
  }
  const int esize = F8 ? 1 : 2;
  TcArgs a{};
  a.wait_ns = wait_budget_ns();
  a.hold_first = test_stall();
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
  const int a_bytes = kBM * kBKBytes, b_bytes = Nt * kBKBytes;
  const int stage_bytes = a_bytes + b_bytes + (W4 ? 1024 : MX ? 2048 : 0);
  a.stages = std::min(8, (kSmemLimit - 1024 - kFixedSmem) / stage_bytes);
  if (a.stages < 2) return cudaErrorInvalidValue;
  if (W4 || MX) {
    // accumulators at columns 0 and buf_cols, then the hidden side's scale
    // factors (w4: one slot of 1s; mxfp8: a slot of 8 columns per stage), then
    // the weight scale factors (a slot of 8 columns per stage)
    a.buf_cols = uint32_t(Nt + 31) / 32 * 32;
    a.tmem_cols = 512;
    auto fits = [&](int stages) {
      const uint32_t sfb_cols = MX ? uint32_t(kSfaSlot * stages) : uint32_t(kSfbCols);
      return 2 * a.buf_cols + sfb_cols + kSfaSlot * stages <= a.tmem_cols;
    };
    while (a.stages > 2 && !fits(a.stages)) --a.stages;
    if (!fits(a.stages)) return cudaErrorInvalidValue;
    a.sfb_col = 2 * a.buf_cols;
    a.sfa_col = a.sfb_col + (MX ? kSfaSlot * a.stages : kSfbCols);
  } else {
    a.tmem_cols = Nt <= 128 ? 256 : 512;
    a.buf_cols = a.tmem_cols / 2;
  }
  const size_t smem = 1024 + size_t(a.stages) * stage_bytes + kFixedSmem;

  CUtensorMap tmW, tmH;
  if (!encode_kmajor(&tmH, hidden, n.N, d.D, Nt, esize)) return cudaErrorInvalidValue;
  if (W4) {
    // the code region covers whole tiles: ceil(V / 128) * 128 rows of
    // ceil(D / 128) * 128 codes; the scale-factor region follows it
    const int rows = plan.vtiles * kBM, kd = a.nkb * 128;
    if (!encode_w4_codes(&tmW, w_lm, rows, kd)) return cudaErrorInvalidValue;
    a.w_sf = static_cast<const uint8_t*>(w_lm) + size_t(rows) * (kd / 2);
  } else if (!encode_kmajor(&tmW, w_lm, n.V, d.D, kBM, esize)) {
    return cudaErrorInvalidValue;
  }
  if (MX) {
    a.w_sf = w_sf;
    a.h_sf = h_sf;
  }
  cudaError_t e = cudaFuncSetAttribute(lmhead_tc_kernel<FMT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  int sms = sm_count();
  if (d.max_sms > 0) sms = std::min(sms, d.max_sms);
  const int grid = std::max(1, std::min(a.units, sms));
  return launch_pdl(lmhead_tc_kernel<FMT>, dim3(grid), dim3(kThreads), smem, st,
                    tmW, tmH, a);
}

}  // namespace

cudaError_t launch_lmhead_tc(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const void* hidden, const void* w_lm, void* ws, int* status,
                             cudaStream_t st) {
  return launch_head<kFmtBf16>(lay, d, plan, hidden, nullptr, w_lm, nullptr, ws, status, st);
}

cudaError_t launch_lmhead_e4m3(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                               const uint8_t* h_q, const float* h_scale, const uint8_t* w_q,
                               const float* w_scale, void* ws, int* status, cudaStream_t st) {
  return launch_head<kFmtE4m3>(lay, d, plan, h_q, h_scale, w_q, w_scale, ws, status, st);
}

cudaError_t launch_lmhead_mx(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const uint8_t* h_q, const uint8_t* h_sf, const uint8_t* w_q,
                             const uint8_t* w_sf, void* ws, int* status, cudaStream_t st) {
  return launch_head<kFmtMx8>(lay, d, plan, h_q, nullptr, w_q, nullptr, ws, status, st, w_sf,
                              h_sf);
}

void mx_token_tiling(int N, int* Nt, int* n_tt) {
  int tt = (N + kMaxNtBs - 1) / kMaxNtBs;
  const int nt = ((N + tt - 1) / tt + 15) / 16 * 16;
  *Nt = nt;
  *n_tt = (N + nt - 1) / nt;
}

cudaError_t launch_lmhead_w4(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const uint8_t* h_q, const float* h_scale, const uint8_t* w4,
                             const float* w_scale, void* ws, int* status, cudaStream_t st) {
  return launch_head<kFmtW4>(lay, d, plan, h_q, h_scale, w4, w_scale, ws, status, st);
}

}  // namespace jet
