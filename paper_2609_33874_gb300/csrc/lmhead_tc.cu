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
// the e4m3 bytes. It keeps three rings: hidden-state tiles and 4-bit weight
// tiles (128 rows x 128 codes and their exponents, 8,704 bytes, one TMA box of
// the pre-tiled buffer), both issued by the producer as far ahead as they
// fit, and two widened e4m3 weight tiles that only live from their
// conversion to their MMA. Eight converter warps (warps 6..13, a
// thread per vocabulary row and half slice) widen every code to the e4m3 value
// 2^e value(code) - exact, since e >= -5 keeps it a normal e4m3 number - into
// the same 128-byte-swizzled operand tile the e4m3 instantiation loads by TMA.
// The MMA, the scales and the epilogue are the e4m3 instantiation's.
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
constexpr int kThreadsW4 = 448;     // + eight converter warps
constexpr int kConvWarps = 8;
constexpr int kMaxRawSlots = 12;
constexpr int kW4TileRows = kW4TileBytes / 128;  // 68
constexpr int kRawBytes = 9216;     // one w4 tile (8,704 bytes) rounded up to 1 KB
enum { kFmtBf16 = 0, kFmtE4m3 = 1, kFmtW4 = 2 };
constexpr int kMaxNt = 256;
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
  const uint8_t* w4;     // w4: tiled codes and exponents
  int* status;
  int N, T, V, D;
  int Nt, n_tt, units, nkb, stages, vtiles;
  int raw_slots;         // w4: 4-bit weight tiles in flight
  int a_slots;           // w4: widened weight tiles
  uint32_t tmem_cols;
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

// Widen blocks 2 h and 2 h + 1 of row r of a landed w4 tile into the e4m3
// operand tile (128-byte swizzle: row r at (r / 8) KB + (r % 8) 128 B, 16-byte
// chunk j in slot j ^ (r % 8)). Per 32-element block: the e4m3 codes of
// 2^e x {0, .5, 1, 1.5, 2, 3, 4, 6} are ((e + 7) << 3) + {-, -8, 0, 4, 8, 12,
// 16, 20} (0 for the zero code), an 8-entry byte table that prmt indexes by
// the 3 magnitude bits of 4 nibbles at a time. The stored sign bits are
// permuted so that the word's bits 7, 15, 23, 31 are the signs of its
// elements 0..3 and bits 3, 11, 19, 27 those of elements 4..7.
__device__ __forceinline__ void widen_w4_row(const uint8_t* raw, uint8_t* A, int r, int h) {
  const uint32_t ex = *reinterpret_cast<const uint32_t*>(raw + kW4CodeBytes + r * 4);
  uint8_t* row = A + (r >> 3) * 1024 + (r & 7) * 128;
#pragma unroll
  for (int c = 2 * h; c < 2 * h + 2; ++c) {
    const uint4 q = *reinterpret_cast<const uint4*>(raw + r * 64 + 16 * (c ^ ((r >> 1) & 3)));
    const uint32_t base = uint32_t(int(int8_t(uint8_t(ex >> (8 * c)))) + 7) << 3;
    // bytes {0, base - 8, base, base + 4} and {base + 8, + 12, + 16, + 20}
    const uint32_t lo = base * 0x01010100u + 0x03FFF800u;
    const uint32_t hi = base * 0x01010101u + 0x14100C08u;
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
    uint32_t o[8];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t m = w[i] & 0x77777777u;
      o[2 * i] = __byte_perm(lo, hi, m) | (w[i] & 0x80808080u);
      o[2 * i + 1] = __byte_perm(lo, hi, m >> 16) | ((w[i] << 4) & 0x80808080u);
    }
    *reinterpret_cast<uint4*>(row + 16 * ((2 * c) ^ (r & 7))) = make_uint4(o[0], o[1], o[2], o[3]);
    *reinterpret_cast<uint4*>(row + 16 * ((2 * c + 1) ^ (r & 7))) =
        make_uint4(o[4], o[5], o[6], o[7]);
  }
}

template <int FMT>
__global__ void __launch_bounds__(FMT == kFmtW4 ? kThreadsW4 : kThreads, 1)
lmhead_tc_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmH,
                 const TcArgs a) {
  constexpr bool F8 = FMT != kFmtBf16;   // e4m3 operands in the MMA
  constexpr bool W4 = FMT == kFmtW4;     // weights widened on chip from 4-bit codes
  constexpr int kBKe = F8 ? kBKBytes : kBK;  // elements of one K slice
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t a_bytes = kBM * 128, b_bytes = uint32_t(a.Nt) * 128;
  // a stage holds the weight and hidden tiles of one K slice; for w4 it holds
  // the hidden tile only, the weights going through the rings after it
  const uint32_t stage_bytes = W4 ? b_bytes : a_bytes + b_bytes;
  uint8_t* aring = smem + size_t(a.stages) * stage_bytes;             // w4: widened tiles
  uint8_t* rawb = aring + (W4 ? size_t(a.a_slots) * a_bytes : 0);     // w4: 4-bit tiles
  float2* red = reinterpret_cast<float2*>(rawb + (W4 ? size_t(a.raw_slots) * kRawBytes : 0));
  int4* hits = reinterpret_cast<int4*>(red + 4 * kMaxNt);                          // [128]
  float* hs = reinterpret_cast<float*>(hits + 128);                                // [256]
  uint64_t* full = reinterpret_cast<uint64_t*>(hs + kMaxNt);
  uint64_t* empty = full + a.stages;
  uint64_t* conv = empty + a.stages;     // w4: a widened tile is ready
  uint64_t* aempty = conv + a.a_slots;   // w4: ... has been consumed by its MMAs
  uint64_t* raw_full = aempty + a.a_slots;  // w4: a 4-bit tile has landed
  uint64_t* raw_empty = raw_full + a.raw_slots;  // w4: ... has been widened
  uint64_t* tfull = raw_empty + a.raw_slots;
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
    for (int s = 0; s < a.a_slots; ++s) {
      mbar_init(conv + s, kConvWarps);
      mbar_init(aempty + s, 1);
    }
    for (int s = 0; s < a.raw_slots; ++s) {
      mbar_init(raw_full + s, 1);
      mbar_init(raw_empty + s, kConvWarps);
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
    if (lane == 0 && W4) {
      // per K slice, in order: the 4-bit weight tile into its ring, then the
      // hidden tile into the stage
      const uint64_t pol_w = policy_evict_first(), pol_h = policy_evict_last();
      int s = 0, sr = 0;
      uint32_t ph = 0, rph = 0, issued = 0, issued_par = 0, rissued = 0, rissued_par = 0;
      bool ok = true, hold = a.hold_first != 0;
      for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
        const int vt = u / a.n_tt, t0 = (u % a.n_tt) * a.Nt;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(raw_empty + sr, rph ^ 1u, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          // the tile is 68 rows of 128 bytes of the w4 buffer's 2-D view
          mbar_arrive_expect_tx(raw_full + sr, kW4TileBytes);
          tma_load_2d(rawb + size_t(sr) * kRawBytes, &tmW, raw_full + sr, 0,
                      (vt * a.nkb + kb) * kW4TileRows, pol_w);
          rissued |= 1u << sr;
          rissued_par = (rissued_par & ~(1u << sr)) | (rph << sr);
          if (++sr == a.raw_slots) {
            sr = 0;
            rph ^= 1u;
          }
          if (!mbar_wait(empty + s, ph ^ 1u, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          if (hold) {
            hold = false;  // test hook: this stage never fills
          } else {
            mbar_arrive_expect_tx(full + s, b_bytes);
            tma_load_2d(smem + size_t(s) * stage_bytes, &tmH, full + s, kb * kBKe, t0, pol_h);
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
        for (int t = 0; t < a.raw_slots; ++t)
          if (rissued & (1u << t))
            mbar_wait(raw_full + t, (rissued_par >> t) & 1u, kDrainNs, nullptr);
        for (int t = 0; t < a.stages; ++t)
          if (issued & (1u << t)) mbar_wait(full + t, (issued_par >> t) & 1u, kDrainNs, nullptr);
      }
    } else if (lane == 0) {
      const uint64_t pol_w = policy_evict_first(), pol_h = policy_evict_last();
      int s = 0;
      uint32_t ph = 0, issued = 0, issued_par = 0;
      bool ok = true, hold = a.hold_first != 0;
      for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
        const int v0 = (u / a.n_tt) * kBM, t0 = (u % a.n_tt) * a.Nt;
        for (int kb = 0; kb < a.nkb; ++kb) {
          if (!mbar_wait(empty + s, ph ^ 1u, a.wait_ns, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + size_t(s) * stage_bytes;
          if (hold) {
            hold = false;  // test hook: this stage never fills
          } else {
            mbar_arrive_expect_tx(full + s, stage_bytes);
            tma_load_2d(sa, &tmW, full + s, kb * kBKe, v0, pol_w);
            tma_load_2d(sa + a_bytes, &tmH, full + s, kb * kBKe, t0, pol_h);
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
      int s = 0, local = 0, ia = 0;
      uint32_t ph = 0, aph = 0;
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
          if (!mbar_wait(full + s, ph, a.wait_ns, abort_flag) ||
              (W4 && !mbar_wait(conv + ia, aph, a.wait_ns, abort_flag))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ss = smem_u32(smem + size_t(s) * stage_bytes);
          const uint32_t sa = W4 ? smem_u32(aring + size_t(ia) * a_bytes) : ss;
          const uint32_t sb = W4 ? ss : ss + a_bytes;
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
          if (W4) {
            mma_commit(aempty + ia);  // ... and the widened tile
            if (++ia == a.a_slots) {
              ia = 0;
              aph ^= 1u;
            }
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
  } else if (W4 && warp >= 6) {
    // ------------------------------------------------------------ w4 converter
    const int r = (threadIdx.x - 192) & (kBM - 1);  // vocabulary row of the tile
    const int hh = (threadIdx.x - 192) >> 7;         // which half of the K slice
    int ia = 0, slot = 0;
    uint32_t aph = 0, rph = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
      for (int kb = 0; kb < a.nkb; ++kb) {
        // one lane waits for the tile and the free slot; __syncwarp orders the
        // other lanes' reads and writes after its wait
        bool got = true;
        if (lane == 0)
          got = mbar_wait(raw_full + slot, rph, a.wait_ns, abort_flag) &&
                mbar_wait(aempty + ia, aph ^ 1u, a.wait_ns, abort_flag);
        if (!__shfl_sync(0xffffffffu, got, 0)) {
          ok = false;
          break;
        }
        __syncwarp();
        widen_w4_row(rawb + size_t(slot) * kRawBytes, aring + size_t(ia) * a_bytes, r, hh);
        fence_proxy_async_shared();  // the widened tile is read by the tensor core
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(conv + ia);
          mbar_arrive(raw_empty + slot);
        }
        if (++ia == a.a_slots) {
          ia = 0;
          aph ^= 1u;
        }
        if (++slot == a.raw_slots) {
          slot = 0;
          rph ^= 1u;
        }
      }
    }
    if (!ok) {
      *abort_flag = 1;
      if (lane == 0) flag(a.status, JET_ERR_TIMEOUT);
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

// the tiled w4 buffer as a [tiles * 68, 128] byte matrix, one tile per box
bool encode_w4_tiles(CUtensorMap* map, const void* base, int tiles) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {128, cuuint64_t(tiles) * kW4TileRows};
  const cuuint64_t strides[1] = {128};
  const cuuint32_t box[2] = {128, cuuint32_t(kW4TileRows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
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
// or tiled 4-bit weights, per-row weight scales and per-token hidden scales
template <int FMT>
cudaError_t launch_head(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                        const void* hidden, const float* h_scale, const void* w_lm,
                        const float* w_scale, void* ws, int* status, cudaStream_t st) {
  constexpr bool F8 = FMT != kFmtBf16, W4 = FMT == kFmtW4;
  const jet_sizes& n = lay.n;
  int n_tt = (n.N + kMaxNt - 1) / kMaxNt;
  const int Nt = ((n.N + n_tt - 1) / n_tt + 15) / 16 * 16;
  n_tt = (n.N + Nt - 1) / Nt;
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
  a.w4 = W4 ? static_cast<const uint8_t*>(w_lm) : nullptr;
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
  const int a_bytes = kBM * kBKBytes, b_bytes = Nt * kBKBytes;
  int room = kSmemLimit - 1024 - kFixedSmem;
  int stage_bytes = a_bytes + b_bytes;
  a.raw_slots = a.a_slots = 0;
  if (W4) {
    // two widened tiles; the rest split between hidden tiles and 4-bit tiles
    stage_bytes = b_bytes;
    a.a_slots = 2;
    room -= a.a_slots * a_bytes;
    a.stages = std::min(8, room / (b_bytes + kRawBytes));
    a.raw_slots = std::min(kMaxRawSlots, (room - a.stages * b_bytes) / kRawBytes);
    if (a.stages < 2 || a.raw_slots < 2) return cudaErrorInvalidValue;
  } else {
    a.stages = std::min(8, room / stage_bytes);
  }
  const size_t smem = 1024 + size_t(a.stages) * stage_bytes + size_t(a.a_slots) * a_bytes +
                      size_t(a.raw_slots) * kRawBytes + kFixedSmem;

  CUtensorMap tmW, tmH;
  if (!encode_kmajor(&tmH, hidden, n.N, d.D, Nt, esize)) return cudaErrorInvalidValue;
  if (W4) {
    if (!encode_w4_tiles(&tmW, w_lm, plan.vtiles * a.nkb)) return cudaErrorInvalidValue;
  } else if (!encode_kmajor(&tmW, w_lm, n.V, d.D, kBM, esize)) {
    return cudaErrorInvalidValue;
  }
  cudaError_t e = cudaFuncSetAttribute(lmhead_tc_kernel<FMT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  int sms = sm_count();
  if (d.max_sms > 0) sms = std::min(sms, d.max_sms);
  const int grid = std::max(1, std::min(a.units, sms));
  return launch_pdl(lmhead_tc_kernel<FMT>, dim3(grid), dim3(W4 ? kThreadsW4 : kThreads), smem, st,
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

cudaError_t launch_lmhead_w4(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const uint8_t* h_q, const float* h_scale, const uint8_t* w4,
                             const float* w_scale, void* ws, int* status, cudaStream_t st) {
  return launch_head<kFmtW4>(lay, d, plan, h_q, h_scale, w4, w_scale, ws, status, st);
}

}  // namespace jet
