// Prefix part of the cascade attention on the 5th-generation tensor cores
// (Sec. 4.1, Fig. 1 "KV-cache text models"; bf16 inputs, f32 accumulation).
//
// One CTA owns one (request r, key/value head kh, prefix chunk, query block):
// the query block is up to 128 query vectors (row, head) of the request's
// group kh, i.e. all candidates' rows share every prefix K/V tile the CTA
// streams - the prefix is read once per group, not once per candidate.
//
//   warp 0      TMA producer: 64-key K and V tiles (d/64 boxes each, 128-byte
//               swizzled) into a 2-stage ring
//   warp 1      TMEM allocator, MMA issuer:
//                 S_j  = Q K_j^T   (M 128 vectors, N 64 keys, K d)   -> TMEM
//                 O   += P_j V_j   (M 128 vectors, N d, K 64 keys)   -> TMEM
//               V_j is the MN-major B operand (d contiguous in memory).
//   warps 2..5  softmax: thread = query vector = TMEM lane. Reads S_j, keeps a
//               running max m and sum l in base 2, writes P_j = 2^(s - m) as
//               bf16 into a 128-byte-swizzled shared tile; O is rescaled in
//               TMEM only when the row max grows by more than 8 (a factor 256),
//               so P stays <= 256 and rescales are rare.
// The CTA writes its unnormalised O and (m, l) as a partial; the merge kernel
// combines the chunks with the candidates' own causal keys.
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

constexpr int kBV = 128;      // query vectors per CTA (MMA M, TMEM lanes)
constexpr int kBN = 64;       // keys per tile
constexpr int kStages = 2;
constexpr int kThreads = 192;
constexpr uint64_t kWaitNs = 2000000000ull;
constexpr uint64_t kDrainNs = 200000000ull;
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the max grows by > 2^8
constexpr int kPrefetch = 4;         // key tiles prefetched into L2 ahead of the TMA loads

template <int DH>
struct Geo {
  static constexpr int kSlices = DH / 64;                   // 64-wide d slices
  static constexpr uint32_t kQBytes = kBV * DH * 2;         // query block
  static constexpr uint32_t kKVBytes = kBN * DH * 2;        // one K (or V) tile
  static constexpr uint32_t kPBytes = kBV * kBN * 2;        // one P tile
  static constexpr uint32_t kOffK = kQBytes;                // stage s: K at kOffK + s * 2 kKV
  static constexpr uint32_t kOffP = kQBytes + kStages * 2 * kKVBytes;
  static constexpr uint32_t kOffBar = kOffP + 2 * kPBytes;
  static constexpr uint32_t kBytes = kOffBar + 256;
  static constexpr uint32_t kTmemCols = (2 * kBN + DH) <= 256 ? 256 : 512;
  static constexpr uint32_t kOCol = 2 * kBN;                // O after the two S buffers
};

struct AttArgs {
  const int32_t* prefix_offset;
  const int32_t* row_offset;
  const int32_t* row_cand;
  const int32_t* cand_row_offset;
  const __nv_bfloat16* q;
  __nv_bfloat16* o;  // final output, written directly by single-chunk requests
  float* o_part;
  float2* ml_part;
  int* status;
  int R, N, C, total_prefix, Hq, Hkv, chunk;
  int has_cand;      // the batch has fed candidate tokens (F > 0)
  float scale_log2;  // log2(e) / sqrt(d)
};

// SW128 K-major position of 16-byte chunk c of row i inside one 64-wide slice
__device__ __forceinline__ uint32_t sw128(int i, int c) {
  return uint32_t(i) * 128u + (uint32_t(c ^ (i & 7)) << 4);
}

// descriptor of an MN-major operand tile written by TMA with 128-byte
// swizzling: 64-element (128-byte) rows along K, slices of 64 MN elements
// `lbo` bytes apart, 8-row groups along K 1024 bytes apart
__device__ __forceinline__ uint64_t desc_mn_sw128(uint32_t addr, uint32_t lbo) {
  uint64_t d = 0;
  d |= uint64_t((addr >> 4) & 0x3FFFu);
  d |= uint64_t((lbo >> 4) & 0x3FFFu) << 16;
  d |= uint64_t(1024 >> 4) << 32;
  d |= uint64_t(1) << 46;
  d |= uint64_t(2) << 61;
  return d;
}

__device__ __forceinline__ void tmem_st_32cols(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(
          taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
      "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
      "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
      "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
      "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
      "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// 3-D TMA load: box {64 d, 1 head, 64 keys} at (x = d, y = head, z = key)
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, uint64_t* bar,
                                            int32_t x, int32_t y, int32_t z, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)),
      "l"(policy)
      : "memory");
}

// 3-D TMA prefetch of the same box into L2 only
__device__ __forceinline__ void tma_prefetch_3d(const CUtensorMap* map, int32_t x, int32_t y,
                                                int32_t z) {
  asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(
                   reinterpret_cast<uint64_t>(map)),
               "r"(x), "r"(y), "r"(z)
               : "memory");
}

template <int DH>
__global__ void __launch_bounds__(kThreads, 1)
attend_prefix_tc_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmK,
                        const __grid_constant__ CUtensorMap tmV,
                        const __grid_constant__ CUtensorMap tmKc,
                        const __grid_constant__ CUtensorMap tmVc, const AttArgs a) {
  using G = Geo<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  // K and V of a stage fill and drain separately: K is free once S_j has been
  // computed, V only after P_j V_j
  uint64_t* k_full = reinterpret_cast<uint64_t*>(smem + G::kOffBar);
  uint64_t* k_empty = k_full + kStages;
  uint64_t* v_full = k_empty + kStages;
  uint64_t* v_empty = v_full + kStages;
  uint64_t* s_full = v_empty + kStages;    // [2]
  uint64_t* s_free = s_full + 2;           // [2]
  uint64_t* p_full = s_free + 2;           // [2]
  uint64_t* p_free = p_full + 2;           // [2]
  uint64_t* q_full = p_free + 2;
  uint64_t* drain = q_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  // query blocks are the slowest grid dimension: blocks past a request's
  // vectors (only long requests have them) come last and exit at once
  const int split = blockIdx.x, qb = blockIdx.z;
  const int r = blockIdx.y / a.Hkv, kh = blockIdx.y % a.Hkv;
  const int g = a.Hq / a.Hkv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (r >= a.R) return;
  const int n0 = a.row_offset[r], nr = a.row_offset[r + 1] - n0;
  const int p0 = a.prefix_offset[r], P = a.prefix_offset[r + 1] - p0;
  if (n0 < 0 || nr < 1 || n0 + nr > a.N || p0 < 0 || P < 0 || p0 + P > a.total_prefix) {
    if (threadIdx.x == 0) flag(a.status, JET_ERR_DEVICE);
    return;
  }
  // a query block holds whole rows: rb rows x g heads (<= 128 vectors)
  const int rb = kBV / g;
  const int row0 = qb * rb;  // first row of the block within the request
  if (row0 >= nr) return;
  const int vbase = row0 * g;
  const int nv = min(rb, nr - row0) * g;
  const int k_begin = split * a.chunk;
  const int k_end = min(P, k_begin + a.chunk);
  const int npt = k_end > k_begin ? (k_end - k_begin + kBN - 1) / kBN : 0;  // prefix tiles
  // the request's last chunk also takes its candidates' own keys: the F_r fed
  // tokens, as extra 64-key tiles masked per row to the row's candidate and
  // position (Sec. 4.1: a candidate attends to its own earlier tokens only)
  const int splits_r = (P + a.chunk - 1) / a.chunk;
  const bool last = npt > 0 && split == splits_r - 1;
  const int f_begin = n0 - r;     // fed-token index of the request's first fed row
  const int F_r = nr - 1;
  const int nct = (last && a.has_cand && F_r > 0) ? (F_r + kBN - 1) / kBN : 0;
  const int ntiles = npt + nct;

  if (npt == 0) {  // an empty chunk: an empty partial
    for (int i = threadIdx.x; i < nv; i += blockDim.x) {
      const int gv = vbase + i;
      const size_t base = (size_t(split) * a.N + n0 + gv / g) * a.Hq + kh * g + gv % g;
      a.ml_part[base] = make_float2(-INFINITY, 0.f);
    }
    return;
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(k_full + s, 1);
      mbar_init(k_empty + s, 1);
      mbar_init(v_full + s, 1);
      mbar_init(v_empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full + b, 1);
      mbar_init(s_free + b, 4);
      mbar_init(p_full + b, 4);
      mbar_init(p_free + b, 1);
    }
    mbar_init(q_full, 5);  // the query TMA (with its bytes) + 4 softmax warps
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, G::kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    if (nct > 0) {
      tma_prefetch_desc(&tmKc);
      tma_prefetch_desc(&tmVc);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      // the query block: rb rows x g heads x d of the request's group kh
      mbar_arrive_expect_tx(q_full, uint32_t(G::kSlices) * 64 * 2 * g * rb);
#pragma unroll
      for (int sl = 0; sl < G::kSlices; ++sl)
        tma_load_3d(smem + sl * (kBV * 128), &tmQ, q_full, sl * 64, kh * g, n0 + row0,
                    policy_evict_first());
      // K_j and V_j are issued as soon as their slots drain, whichever first
      const uint64_t pol = policy_evict_first();
      uint32_t k_issued = 0, k_par = 0, v_issued = 0, v_par = 0;
      int jk = 0, jv = 0;
      bool ok = true;
      uint64_t t_last = global_timer_ns();
      while (jv < ntiles) {
        bool progressed = false;
        if (jk < ntiles) {
          const int s = jk % kStages;
          const uint32_t ph = (jk / kStages) & 1;
          if (mbar_test(k_empty + s, ph ^ 1u)) {
            uint8_t* ks = smem + G::kOffK + s * 2 * G::kKVBytes;
            mbar_arrive_expect_tx(k_full + s, G::kKVBytes);
            const bool pre = jk < npt;
            const CUtensorMap* mk = pre ? &tmK : &tmKc;
            const int key = pre ? p0 + k_begin + jk * kBN : f_begin + (jk - npt) * kBN;
#pragma unroll
            for (int sl = 0; sl < G::kSlices; ++sl)
              tma_load_3d(ks + sl * (kBN * 128), mk, k_full + s, sl * 64, kh, key, pol);
            // keep kPrefetch further tiles on their way into L2: two shared
            // stages alone hold too few bytes in flight to cover HBM latency
            for (int jp = (jk == 0 ? 1 : jk + kPrefetch); jp <= jk + kPrefetch && jp < npt;
                 ++jp) {
              const int kp = p0 + k_begin + jp * kBN;
#pragma unroll
              for (int sl = 0; sl < G::kSlices; ++sl) {
                tma_prefetch_3d(&tmK, sl * 64, kh, kp);
                tma_prefetch_3d(&tmV, sl * 64, kh, kp);
              }
            }
            k_issued |= 1u << s;
            k_par = (k_par & ~(1u << s)) | (ph << s);
            ++jk;
            progressed = true;
          }
        }
        if (jv < jk) {
          const int s = jv % kStages;
          const uint32_t ph = (jv / kStages) & 1;
          if (mbar_test(v_empty + s, ph ^ 1u)) {
            uint8_t* vs = smem + G::kOffK + s * 2 * G::kKVBytes + G::kKVBytes;
            mbar_arrive_expect_tx(v_full + s, G::kKVBytes);
            const bool pre = jv < npt;
            const CUtensorMap* mv = pre ? &tmV : &tmVc;
            const int key = pre ? p0 + k_begin + jv * kBN : f_begin + (jv - npt) * kBN;
#pragma unroll
            for (int sl = 0; sl < G::kSlices; ++sl)
              tma_load_3d(vs + sl * (kBN * 128), mv, v_full + s, sl * 64, kh, key, pol);
            v_issued |= 1u << s;
            v_par = (v_par & ~(1u << s)) | (ph << s);
            ++jv;
            progressed = true;
          }
        }
        const uint64_t now = global_timer_ns();
        if (progressed) {
          t_last = now;
        } else if (*abort_flag || now - t_last > kWaitNs) {
          ok = false;
          break;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        // let every copy already issued land before the CTA can exit
        for (int t = 0; t < kStages; ++t) {
          if (k_issued & (1u << t)) mbar_wait(k_full + t, (k_par >> t) & 1u, kDrainNs, nullptr);
          if (v_issued & (1u << t)) mbar_wait(v_full + t, (v_par >> t) & 1u, kDrainNs, nullptr);
        }
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t id_s = idesc_bf16_f32(kBV, kBN);
      const uint32_t id_o = idesc_bf16_f32(kBV, DH) | (1u << 16);  // B (V) is MN-major
      const uint32_t qs = smem_u32(smem);
      bool ok = mbar_wait(q_full, 0, kWaitNs, abort_flag);
      tc_fence_after();
      // issue S_j = Q K_j^T and O += P_j V_j in whichever order their inputs
      // become ready; S_j always precedes P_j V_j
      int js = 0, jo = 0;
      uint64_t t_last = global_timer_ns();
      while (ok && jo < ntiles) {
        bool progressed = false;
        if (js < ntiles) {
          const int s = js % kStages, b = js & 1;
          if (mbar_test(k_full + s, (js / kStages) & 1) &&
              mbar_test(s_free + b, ((js >> 1) & 1) ^ 1u)) {
            tc_fence_after();
            const uint32_t ks = smem_u32(smem + G::kOffK + s * 2 * G::kKVBytes);
#pragma unroll
            for (int st = 0; st < DH / 16; ++st) {
              const int sl = st >> 2, k = st & 3;
              mma_f16(tmem + b * kBN, desc_k_sw128(qs + sl * (kBV * 128) + 32 * k),
                      desc_k_sw128(ks + sl * (kBN * 128) + 32 * k), id_s, st != 0);
            }
            mma_commit(s_full + b);
            mma_commit(k_empty + s);
            ++js;
            progressed = true;
          }
        }
        if (jo < js) {
          const int s = jo % kStages, b = jo & 1;
          if (mbar_test(p_full + b, (jo >> 1) & 1) && mbar_test(v_full + s, (jo / kStages) & 1)) {
            tc_fence_after();
            const uint32_t ps = smem_u32(smem + G::kOffP + b * G::kPBytes);
            const uint32_t vs = smem_u32(smem + G::kOffK + s * 2 * G::kKVBytes + G::kKVBytes);
#pragma unroll
            for (int k = 0; k < kBN / 16; ++k)
              mma_f16(tmem + G::kOCol, desc_k_sw128(ps + 32 * k),
                      desc_mn_sw128(vs + k * 16 * 128, kBN * 128), id_o, (jo | k) != 0);
            mma_commit(p_free + b);
            mma_commit(v_empty + s);
            ++jo;
            progressed = true;
          }
        }
        const uint64_t now = global_timer_ns();
        if (progressed) {
          t_last = now;
        } else if (*abort_flag || now - t_last > kWaitNs) {
          ok = false;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        mma_commit(drain);
        mbar_wait(drain, 0, kDrainNs, nullptr);
      }
    }
  } else {
    // ---------------------------------------------------------------- softmax
    const int q4 = warp & 3;
    const int i = q4 * 32 + lane;  // query vector within the block = TMEM lane
    const uint32_t lane_off = uint32_t(q4 * 32) << 16;
    const bool valid = i < nv;
    int n = 0, h = 0;
    int fa = 1, fb = 0;  // fed-token indices this vector may see (none: shared row)
    if (valid) {
      const int gv = vbase + i;
      n = n0 + gv / g;
      h = kh * g + gv % g;
      const int c = a.row_cand[n];
      if (c >= 0 && c < a.C) {
        fa = a.cand_row_offset[c] - r - 1;  // y_{c,1}
        fb = n - r - 1;                     // the row's own fed token, inclusive
      }
    }
    // the query block arrives by TMA (rows [0, rb g)); zero the rows past it
    // so that no stale shared memory enters the MMA
    {
      if (i >= rb * g) {
#pragma unroll
        for (int c = 0; c < DH / 8; ++c)
          *reinterpret_cast<uint4*>(smem + (c >> 3) * (kBV * 128) + sw128(i, c & 7)) =
              make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_full);
    }
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      const int b = j & 1;
      if (!warp_mbar_wait(s_full + b, (j >> 1) & 1, kWaitNs, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float sv[kBN];
      {
        float t0[32], t1[32];
        tmem_ld_32cols(tmem + lane_off + b * kBN, t0);
        tmem_ld_32cols(tmem + lane_off + b * kBN + 32, t1);
        tmem_wait_ld();
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          sv[c] = t0[c];
          sv[c + 32] = t1[c];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(s_free + b);
      // visible keys of this tile: [klo, khi) of its 64 slots
      int klo = 0, khi;
      if (j < npt) {
        khi = min(kBN, k_end - (k_begin + j * kBN));
      } else {
        const int f0 = f_begin + (j - npt) * kBN;
        klo = max(0, fa - f0);
        khi = min(kBN, fb - f0 + 1);
      }
      float mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < kBN; ++c) {
        sv[c] = (c >= klo && c < khi) ? sv[c] * a.scale_log2 : -INFINITY;
        mt = fmaxf(mt, sv[c]);
      }
      // P_j reuses buffer b: PV_{j-2} must be done reading it
      if (j >= 2 && !warp_mbar_wait(p_free + b, ((j - 2) >> 1) & 1, kWaitNs, abort_flag)) {
        ok = false;
        break;
      }
      if (mt > m_used + kRescaleLog2) {
        const float m_new = mt;
        if (j >= 1) {
          // O holds PV_0 .. PV_{j-1}: wait for PV_{j-1}, then rescale it in TMEM
          if (!warp_mbar_wait(p_free + ((j - 1) & 1), ((j - 1) >> 1) & 1, kWaitNs, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float f = ex2(m_used - m_new);
#pragma unroll 1
          for (int c0 = 0; c0 < DH; c0 += 32) {
            float ov[32];
            tmem_ld_32cols(tmem + lane_off + G::kOCol + c0, ov);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < 32; ++c) ov[c] *= f;
            tmem_st_32cols(tmem + lane_off + G::kOCol + c0, ov);
          }
          tmem_wait_st();
          l *= f;
        }
        m_used = m_new;
      }
      // P_j = 2^(s - m_used) as bf16, 128-byte swizzled; the row sum uses the
      // rounded values, which are what the tensor core multiplies
      uint8_t* pb = smem + G::kOffP + b * G::kPBytes;
      float psum = 0.f;
#pragma unroll
      for (int cc = 0; cc < 8; ++cc) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float x0 = ex2(sv[cc * 8 + 2 * e] - m_used);
          const float x1 = ex2(sv[cc * 8 + 2 * e + 1] - m_used);
          w[e] = pack_bf16(x0, x1);
          const __nv_bfloat162 hb = *reinterpret_cast<const __nv_bfloat162*>(&w[e]);
          psum += __bfloat162float(hb.x) + __bfloat162float(hb.y);
        }
        *reinterpret_cast<uint4*>(pb + sw128(i, cc)) = make_uint4(w[0], w[1], w[2], w[3]);
      }
      l += psum;
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full + b);
    }
    // wait for the last PV, then write the partial
    if (ok) {
      const int jl = ntiles - 1;
      ok = warp_mbar_wait(p_free + (jl & 1), (jl >> 1) & 1, kWaitNs, abort_flag);
    }
    if (ok) {
      tc_fence_after();
      const size_t base = (size_t(split) * a.N + n) * a.Hq + h;
      const bool direct = splits_r == 1;  // the whole row in this CTA: final output
      const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
      for (int c0 = 0; c0 < DH; c0 += 32) {
        float ov[32];
        tmem_ld_32cols(tmem + lane_off + G::kOCol + c0, ov);
        tmem_wait_ld();
        if (valid && direct) {
          uint4* dst = reinterpret_cast<uint4*>(a.o + (size_t(n) * a.Hq + h) * DH + c0);
#pragma unroll
          for (int c = 0; c < 4; ++c)
            dst[c] = make_uint4(pack_bf16(ov[8 * c] * inv, ov[8 * c + 1] * inv),
                                pack_bf16(ov[8 * c + 2] * inv, ov[8 * c + 3] * inv),
                                pack_bf16(ov[8 * c + 4] * inv, ov[8 * c + 5] * inv),
                                pack_bf16(ov[8 * c + 6] * inv, ov[8 * c + 7] * inv));
        } else if (valid) {
          float4* dst = reinterpret_cast<float4*>(a.o_part + base * DH + c0);
#pragma unroll
          for (int c = 0; c < 8; ++c)
            dst[c] = make_float4(ov[4 * c], ov[4 * c + 1], ov[4 * c + 2], ov[4 * c + 3]);
        }
      }
      if (valid && !direct) a.ml_part[base] = make_float2(m_used, l);
    } else {
      *abort_flag = 1;
      flag(a.status, JET_ERR_TIMEOUT);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, G::kTmemCols);
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

// packed [keys, Hkv, DH] bf16 K or V: box of 64 d x 1 head x 64 keys
// packed [rows, heads, DH] bf16: box of 64 d x box_heads heads x box_rows rows
bool encode_3d(CUtensorMap* map, const void* base, int rows, int heads, int DH, int box_heads,
               int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {cuuint64_t(DH), cuuint64_t(heads), cuuint64_t(rows)};
  const cuuint64_t strides[2] = {cuuint64_t(DH) * 2, cuuint64_t(heads) * DH * 2};
  const cuuint32_t box[3] = {64, cuuint32_t(box_heads), cuuint32_t(box_rows)};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One warp per (row, query head) of a request whose prefix spans several
// chunks: combine the chunks' base-2 partials (the last chunk also holds the
// candidate's own keys) and normalise. Single-chunk requests were written by
// the attention kernel itself.
template <int DH>
__global__ void __launch_bounds__(256)
attend_combine_kernel(const int32_t* __restrict__ prefix_offset, const int32_t* __restrict__ row_req,
                      int N, int R, int Hq, int chunk, const float* __restrict__ o_part,
                      const float2* __restrict__ ml_part, __nv_bfloat16* __restrict__ o,
                      int* status) {
  const int lane = threadIdx.x & 31;
  const long long idx = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (idx >= (long long)N * Hq) return;
  const int n = int(idx / Hq), h = int(idx % Hq);
  const int r = row_req[n];
  if (r < 0 || r >= R) {
    if (lane == 0) flag(status, JET_ERR_DEVICE);
    return;
  }
  const int P = prefix_offset[r + 1] - prefix_offset[r];
  const int splits_r = (P + chunk - 1) / chunk;
  if (splits_r <= 1) return;
  constexpr int PER = DH / 32;
  float acc[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) acc[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int s = 0; s < splits_r; ++s) {
    const size_t base = (size_t(s) * N + n) * Hq + h;
    const float2 ml = ml_part[base];
    if (!(ml.y > 0.f)) continue;
    const float mn = fmaxf(m, ml.x);
    const float fa = exp2f(m - mn), fb = exp2f(ml.x - mn);
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = acc[i] * fa + o_part[base * DH + lane + 32 * i] * fb;
    l = l * fa + ml.y * fb;
    m = mn;
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
  for (int i = 0; i < PER; ++i)
    o[(size_t(n) * Hq + h) * DH + lane + 32 * i] = __float2bfloat16_rn(acc[i] * inv);
}

template <int DH>
cudaError_t launch_dh(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                      const void* q, const void* k_pre, const void* v_pre, const void* k_cand,
                      const void* v_cand, void* o, float* o_part, float2* ml_part, int* status,
                      cudaStream_t st) {
  const jet_sizes& n = lay.n;
  const int F = n.N - n.R;
  const int g = d.Hq / d.Hkv;
  if (g > kBV) return cudaErrorInvalidValue;
  CUtensorMap tmQ, tmK, tmV, tmKc, tmVc;
  if (!encode_3d(&tmQ, q, n.N, d.Hq, DH, g, kBV / g) ||
      !encode_3d(&tmK, k_pre, n.total_prefix, d.Hkv, DH, 1, kBN) ||
      !encode_3d(&tmV, v_pre, n.total_prefix, d.Hkv, DH, 1, kBN))
    return cudaErrorInvalidValue;
  if (F > 0) {
    if (!encode_3d(&tmKc, k_cand, F, d.Hkv, DH, 1, kBN) ||
        !encode_3d(&tmVc, v_cand, F, d.Hkv, DH, 1, kBN))
      return cudaErrorInvalidValue;
  } else {
    tmKc = tmK;  // never read: no request has candidate tiles
    tmVc = tmV;
  }
  AttArgs a{};
  a.prefix_offset = lay.prefix_offset;
  a.row_offset = lay.row_offset;
  a.row_cand = lay.row_cand;
  a.cand_row_offset = lay.cand_row_offset;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.o = static_cast<__nv_bfloat16*>(o);
  a.o_part = o_part;
  a.ml_part = ml_part;
  a.status = status;
  a.R = n.R;
  a.N = n.N;
  a.C = n.C;
  a.total_prefix = n.total_prefix;
  a.Hq = d.Hq;
  a.Hkv = d.Hkv;
  a.chunk = plan.chunk;
  a.has_cand = F > 0;
  a.scale_log2 = 1.4426950408889634f / sqrtf(float(DH));
  const size_t smem = Geo<DH>::kBytes + 1024;
  cudaError_t e = cudaFuncSetAttribute(attend_prefix_tc_kernel<DH>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(plan.splits, unsigned(n.R * d.Hkv), plan.qgroups);
  attend_prefix_tc_kernel<DH><<<grid, kThreads, smem, st>>>(tmQ, tmK, tmV, tmKc, tmVc, a);
  e = cudaGetLastError();
  if (e != cudaSuccess || plan.splits <= 1) return e;
  const long long warps = (long long)n.N * d.Hq;
  attend_combine_kernel<DH><<<unsigned((warps + 7) / 8), 256, 0, st>>>(
      lay.prefix_offset, lay.row_req, n.N, n.R, d.Hq, plan.chunk, o_part, ml_part,
      static_cast<__nv_bfloat16*>(o), status);
  return cudaGetLastError();
}

}  // namespace

int attn_tc_block() { return kBV; }

cudaError_t launch_attend_tc(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                             const void* q, const void* k_pre, const void* v_pre,
                             const void* k_cand, const void* v_cand, void* o, float* o_part,
                             float2* ml_part, int* status, cudaStream_t st) {
#define JET_TC(DH)                                                                          \
  return launch_dh<DH>(lay, d, plan, q, k_pre, v_pre, k_cand, v_cand, o, o_part, ml_part, \
                       status, st)
  if (d.d == 64) JET_TC(64);
  if (d.d == 128) JET_TC(128);
  if (d.d == 256) JET_TC(256);
#undef JET_TC
  return cudaErrorInvalidValue;
}

}  // namespace jet
