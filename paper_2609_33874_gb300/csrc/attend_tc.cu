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
//               P_j is read from TMEM, V_j is the MN-major B operand (d
//               contiguous in memory).
//   warps 2..5  softmax: thread = query vector = TMEM lane. Reads S_j, keeps a
//               running max m and sum l in base 2, writes P_j = 2^(s - m) as
//               bf16 pairs into its own TMEM lane, where the P V MMA reads it
//               as its A operand (no shared-memory round trip); O is rescaled in
//               TMEM only when the row max grows by more than 8 (a factor 256),
//               so P stays <= 256 and rescales are rare; at the item's end
//               they write its output through shared memory (coalesced).
//   warp 6      scheduler: claims work items one ahead, computes their
//               geometry and starts their query block on the way into L2.
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
constexpr int kThreads = 224;
constexpr int kSchedWarp = 6;  // the work-item scheduler
constexpr uint64_t kDrainNs = 200000000ull;
constexpr float kRescaleLog2 = 8.f;  // rescale O only when the max grows by > 2^8

template <int DH>
struct Geo {
  static constexpr int kSlices = DH / 64;                   // 64-wide d slices
  static constexpr uint32_t kQBytes = kBV * DH * 2;         // query block
  static constexpr uint32_t kKVBytes = kBN * DH * 2;        // one K (or V) tile
  static constexpr uint32_t kOffK = kQBytes;                // stage s: K at kOffK + s * 2 kKV
  // the output stage: 32 rows of 128 bytes per softmax warp
  static constexpr uint32_t kOffStage = kQBytes + kStages * 2 * kKVBytes;
  static constexpr uint32_t kOffBar = kOffStage + 4 * 32 * 128;
  static constexpr uint32_t kBytes = kOffBar + 512;
  // TMEM: the two S buffers, O, then the two P buffers (bf16 pairs, 32 columns)
  static constexpr uint32_t kTmemCols = (2 * kBN + DH + 2 * (kBN / 2)) <= 256 ? 256 : 512;
  static constexpr uint32_t kOCol = 2 * kBN;                // O after the two S buffers
  static constexpr uint32_t kPCol = 2 * kBN + DH;           // P buffer b at kPCol + 32 b
};

struct AttArgs {
  const int32_t* prefix_offset;
  const int32_t* row_offset;
  const int32_t* req_order;
  const int32_t* row_cand;
  const int32_t* cand_row_offset;
  const __nv_bfloat16* q;
  __nv_bfloat16* o;  // final output, written directly by single-chunk requests
  float* o_part;
  float2* ml_part;
  int* status;
  int4* items;       // work list (attend_items_kernel)
  int* item_count;
  int* item_next;    // next item to take (dynamic schedule)
  int R, N, C, total_prefix, Hq, Hkv, chunk;
  int g, rb;         // query heads per kv head; rows per query block (128 / g)
  int sorted;        // 1: take items from the longest-first work list; 0: static
                     // round-robin over all (request, kv head, block, chunk) slots
  int splits;        // chunks per request (the plan's), for the static order
  long long n_all;   // slots in the static order
  int has_cand;      // the batch has fed candidate tokens (F > 0)
  int prefill;       // 1: causal self-attention over the prefixes (rows = prefix positions)
  float scale_log2;  // log2(e) / sqrt(d)
  uint64_t wait_ns;  // budget of one bounded wait (jet_set_wait_budget_ns)
  int hold_first;    // test hook (jet_set_test_stall): withhold the first query block
  int static_only;   // 1: one slot per CTA (the grid covers every slot; no shared counter)
};

// SW128 K-major position of 16-byte chunk c of row i inside one 64-wide slice
__device__ __forceinline__ uint32_t sw128(int i, int c) {
  return uint32_t(i) * 128u + (uint32_t(c ^ (i & 7)) << 4);
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

// A request's P prefix keys in chunks of nearly equal length: at most
// ceil(P / chunk) chunks of a whole number of 64-key tiles each, none empty
// (the last also takes the candidates' own keys).
__device__ __forceinline__ int req_splits(int P, int chunk, int* tiles_per_split) {
  const int tiles = (P + kBN - 1) / kBN;
  const int s0 = max(1, (P + chunk - 1) / chunk);
  const int per = (tiles + s0 - 1) / s0;
  *tiles_per_split = per;
  return (tiles + per - 1) / per;
}

// Geometry of one work item (request r, key/value head kh, query block qb,
// prefix chunk split); every role derives it the same way from the item.
struct ItemGeo {
  int r, kh, n0, nr, p0, P, row0, vbase, nv, k_begin, k_end, npt, nct, ntiles, splits_r, f_begin;
  int split;
  bool ok;
};

__device__ __forceinline__ ItemGeo item_geo(const AttArgs& a, int4 it) {
  ItemGeo e{};
  e.r = it.x;
  e.kh = it.y;
  const int qb = it.z;
  e.split = it.w;
  e.ok = false;
  if (e.r < 0 || e.r >= a.R || e.kh < 0 || e.kh >= a.Hkv) return e;
  if (a.prefill) {
    // prefill: the rows are the request's prefix positions and a block of
    // them sees the keys up to its last position (per-row causal mask in the
    // softmax); one chunk per item, the output written directly
    e.p0 = a.prefix_offset[e.r];
    e.P = a.prefix_offset[e.r + 1] - e.p0;
    if (e.p0 < 0 || e.P < 1 || e.p0 + e.P > a.total_prefix || e.split != 0) return e;
    e.n0 = e.p0;
    e.nr = e.P;
    e.row0 = qb * a.rb;
    if (e.row0 >= e.nr) return e;
    e.vbase = e.row0 * a.g;
    e.nv = min(a.rb, e.nr - e.row0) * a.g;
    e.splits_r = 1;
    e.k_begin = 0;
    e.k_end = min(e.P, e.row0 + a.rb);
    e.npt = (e.k_end + kBN - 1) / kBN;
    e.nct = 0;
    e.f_begin = 0;
    e.ntiles = e.npt;
    e.ok = true;
    return e;
  }
  e.n0 = a.row_offset[e.r];
  e.nr = a.row_offset[e.r + 1] - e.n0;
  e.p0 = a.prefix_offset[e.r];
  e.P = a.prefix_offset[e.r + 1] - e.p0;
  if (e.n0 < 0 || e.nr < 1 || e.n0 + e.nr > a.N || e.p0 < 0 || e.P < 1 ||
      e.p0 + e.P > a.total_prefix)
    return e;
  e.row0 = qb * a.rb;
  if (e.row0 >= e.nr) return e;
  e.vbase = e.row0 * a.g;
  e.nv = min(a.rb, e.nr - e.row0) * a.g;
  int per = 0;
  e.splits_r = req_splits(e.P, a.chunk, &per);
  if (e.split >= e.splits_r) return e;
  e.k_begin = e.split * per * kBN;
  e.k_end = min(e.P, e.k_begin + per * kBN);
  e.npt = (e.k_end - e.k_begin + kBN - 1) / kBN;
  // the request's last chunk also takes its candidates' own keys: the F_r fed
  // tokens, as extra 64-key tiles masked per row to the row's candidate and
  // position (Sec. 4.1: a candidate attends to its own earlier tokens only)
  e.f_begin = e.n0 - e.r;  // fed-token index of the request's first fed row
  const int F_r = e.nr - 1;
  e.nct = (e.split == e.splits_r - 1 && a.has_cand && F_r > 0) ? (F_r + kBN - 1) / kBN : 0;
  e.ntiles = e.npt + e.nct;
  e.ok = true;
  return e;
}

// The work list: every (request, kv head, query block, chunk) that has keys
// and vectors, longest first (counting sort on the tile count), for the
// persistent kernel's dynamic schedule. One block.
constexpr int kBuckets = 256;

constexpr int kItemCache = 16384;  // candidate items whose bucket stays in shared memory

__device__ __forceinline__ int4 item_of(const AttArgs& a, long long idx, int splits) {
  const int split = int(idx % splits);
  const long long rest = idx / splits;
  const int rk = int(rest % (a.R * a.Hkv));
  const int qb = int(rest / (a.R * a.Hkv));
  return make_int4(rk / a.Hkv, rk % a.Hkv, qb, split);
}

__global__ void __launch_bounds__(1024)
attend_items_kernel(const AttArgs a, int qgroups, int splits) {
  pdl_begin();
  __shared__ int hist[kBuckets];
  __shared__ int cursor[kBuckets];
  __shared__ int wsum[kBuckets / 32];
  __shared__ uint8_t bucket[kItemCache];  // 0: no item, else min(tiles, 255)
  for (int b = threadIdx.x; b < kBuckets; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  const long long n_all = (long long)a.R * a.Hkv * qgroups * splits;
  for (long long idx = threadIdx.x; idx < n_all; idx += blockDim.x) {
    const ItemGeo e = item_geo(a, item_of(a, idx, splits));
    const int b = e.ok ? min(e.ntiles, kBuckets - 1) : 0;
    if (idx < kItemCache) bucket[idx] = uint8_t(b);
    if (b > 0) atomicAdd(&hist[b], 1);
  }
  __syncthreads();
  // exclusive scan of the buckets from the longest down (longest items first)
  if (threadIdx.x < kBuckets) {
    const int t = threadIdx.x, lane = t & 31, w = t >> 5;
    const int val = hist[kBuckets - 1 - t];
    int inc = val;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    if (lane == 31) wsum[w] = inc;
    __syncwarp();
    asm volatile("bar.sync 1, %0;" ::"r"(kBuckets) : "memory");
    int base = 0;
    for (int i = 0; i < w; ++i) base += wsum[i];
    cursor[kBuckets - 1 - t] = base + inc - val;
    if (t == kBuckets - 1) {
      *a.item_count = base + inc;
      *a.item_next = 0;
    }
  }
  __syncthreads();
  for (long long idx = threadIdx.x; idx < n_all; idx += blockDim.x) {
    const int4 it = item_of(a, idx, splits);
    int b;
    if (idx < kItemCache) {
      b = bucket[idx];
    } else {
      const ItemGeo e = item_geo(a, it);
      b = e.ok ? min(e.ntiles, kBuckets - 1) : 0;
    }
    if (b > 0) a.items[atomicAdd(&cursor[b], 1)] = it;
  }
}

// The shared item counter of the dynamic schedule starts at zero. The
// layout arrays every work item's geometry is read from are pulled into L2 on
// the way (the LM head's weight stream evicts them between steps), so that
// the attention kernel's first claims do not wait on DRAM.
__global__ void attend_reset_kernel(int* item_next, const int32_t* prefix_offset,
                                    const int32_t* row_offset, const int32_t* req_order,
                                    const int32_t* row_cand, const int32_t* cand_row_offset,
                                    int R, int N, int C) {
  pdl_begin();
  if (threadIdx.x == 0) *item_next = 0;
  auto pull = [](const int32_t* p, int n) {
    for (int i = 32 * int(threadIdx.x); i < n; i += 32 * int(blockDim.x))
      asm volatile("prefetch.global.L2 [%0];" ::"l"(p + i));
  };
  pull(prefix_offset, R + 1);
  pull(row_offset, R + 1);
  if (req_order) pull(req_order, R);
  if (row_cand) pull(row_cand, N);
  if (cand_row_offset) pull(cand_row_offset, C + 1);
}

// The k-th work item of the unsorted order - requests by decreasing prefix
// length (req_order); within a request kv head, query block and chunk, the
// chunk fastest - counting only items that have keys and vectors. One warp
// scans the requests' item counts 32 at a time; false past the last item.
__device__ __forceinline__ bool nth_item(const AttArgs& a, int k, int lane, int4* out) {
  int before = 0;
  for (int base = 0; base < a.R; base += 32) {
    const int ri = base + lane;
    int cnt = 0, r = 0, nq = 0, sp = 0;
    if (ri < a.R) {
      r = a.req_order[ri];
      if (r >= 0 && r < a.R) {
        const int P = a.prefix_offset[r + 1] - a.prefix_offset[r];
        const int nr = a.row_offset[r + 1] - a.row_offset[r];
        int per = 0;
        sp = P >= 1 ? req_splits(P, a.chunk, &per) : 0;
        nq = nr >= 1 ? (nr + a.rb - 1) / a.rb : 0;
        cnt = a.Hkv * nq * sp;
      }
    }
    int inc = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += y;
    }
    const int total = __shfl_sync(0xffffffffu, inc, 31);
    if (k < before + total) {
      const unsigned hit = __ballot_sync(0xffffffffu, k < before + inc);
      const int src = __ffs(hit) - 1;
      const int kk = k - before - __shfl_sync(0xffffffffu, inc - cnt, src);
      r = __shfl_sync(0xffffffffu, r, src);
      nq = __shfl_sync(0xffffffffu, nq, src);
      sp = __shfl_sync(0xffffffffu, sp, src);
      const int split = kk % sp, rest = kk / sp;
      *out = make_int4(r, rest / nq, rest % nq, split);
      return true;
    }
    before += total;
  }
  return false;
}

// One work item as the scheduler warp publishes it: the item and the geometry
// every role needs (16-byte aligned entries: the ring is read with vector loads).
struct __align__(16) RingItem {
  int4 it;
  ItemGeo e;
};
static_assert(sizeof(RingItem) % 16 == 0, "ring entries keep 16-byte alignment");

// One persistent CTA per SM. The scheduler warp claims the work items one
// ahead of the others (the first one without touching the shared counter),
// computes their geometry once and starts their query block on its way into
// L2; the other roles take the items from a two-slot ring and release a slot
// when they are done with its item. All barrier phases run on counters that
// continue across items, so the next item's query block and first K/V tiles
// load while the current item's last tiles and its output are still in flight.
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
  // the item ring first (16-byte aligned entries at a 1024-byte aligned
  // offset), then the barriers. K and V of a stage fill and drain separately:
  // K is free once S_j has been computed, V only after P_j V_j
  RingItem* ring = reinterpret_cast<RingItem*>(smem + G::kOffBar);  // [2]
  uint64_t* k_full = reinterpret_cast<uint64_t*>(ring + 2);
  uint64_t* k_empty = k_full + kStages;
  uint64_t* v_full = k_empty + kStages;
  uint64_t* v_empty = v_full + kStages;
  uint64_t* s_full = v_empty + kStages;    // [2]
  uint64_t* s_free = s_full + 2;           // [2]
  uint64_t* p_full = s_free + 2;           // [2]
  uint64_t* p_free = p_full + 2;           // [2]
  uint64_t* item_full = p_free + 2;        // [2]
  uint64_t* item_empty = item_full + 2;    // [2]
  uint64_t* q_full = item_empty + 2;       // query block of the current item landed
  uint64_t* q_free = q_full + 1;           // last QK^T of the previous item done
  uint64_t* o_free = q_free + 1;           // previous item's O read out of TMEM
  uint64_t* qz_done = o_free + 1;          // unused query rows zeroed (once)
  uint64_t* drain = qz_done + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = a.g, rb = a.rb;
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
      mbar_init(item_full + b, 1);
      mbar_init(item_empty + b, 6);  // producer, MMA thread, 4 softmax warps
    }
    mbar_init(q_full, 1);
    mbar_init(q_free, 1);
    mbar_init(o_free, 4);
    mbar_init(qz_done, 4);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    if (a.has_cand) {
      tma_prefetch_desc(&tmKc);
      tma_prefetch_desc(&tmVc);
    }
  }
  // global memory and TMEM only after the previous kernel of the stream is done
  pdl_begin();
  if (warp == 1) {
    tmem_alloc(tmem_slot, G::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int4 kDone = make_int4(-1, -1, -1, -1);

  if (warp == kSchedWarp) {
    // ---------------------------------------------------------------- scheduler
    const int count = a.sorted ? *a.item_count : 0;
    for (int u = 0;; ++u) {
      const int slot = u & 1;
      bool okw = true;
      if (lane == 0) okw = mbar_wait(item_empty + slot, ((u >> 1) & 1) ^ 1u, a.wait_ns, abort_flag);
      if (!__shfl_sync(0xffffffffu, okw ? 1 : 0, 0)) {
        if (lane == 0) {
          *abort_flag = 1;
          flag(a.status, JET_ERR_TIMEOUT);
        }
        break;
      }
      // the CTA's first item is number blockIdx.x; later ones come from the
      // shared counter, past the grid's first items
      int4 it = kDone;
      ItemGeo e{};
      if (a.sorted) {
        if (lane == 0) {
          for (bool first = (u == 0);; first = false) {
            const int idx = first ? int(blockIdx.x) : int(gridDim.x) + atomicAdd(a.item_next, 1);
            if (idx >= count) break;
            const int4 cand = a.items[idx];
            const ItemGeo ce = item_geo(a, cand);
            if (ce.ok) {
              it = cand;
              e = ce;
              break;
            }
            flag(a.status, JET_ERR_DEVICE);  // the list holds an item the layout lacks
          }
        }
      } else {
        int k = u == 0 ? int(blockIdx.x) : -1;
        if (u > 0 && !a.static_only) {
          if (lane == 0) k = int(gridDim.x) + atomicAdd(a.item_next, 1);
          k = __shfl_sync(0xffffffffu, k, 0);
        }
        int4 cand;
        if (k >= 0 && nth_item(a, k, lane, &cand)) {
          const ItemGeo ce = item_geo(a, cand);
          if (ce.ok) {
            it = cand;
            e = ce;
          } else if (lane == 0) {
            flag(a.status, JET_ERR_DEVICE);
          }
        }
      }
      if (lane == 0) {
        ring[slot].it = it;
        ring[slot].e = e;
        mbar_arrive(item_full + slot);
        // start the query block on its way into L2 (K/V tiles are not
        // prefetched: extra requests in flight only delay the demand loads)
        if (it.x >= 0) {
#pragma unroll
          for (int sl = 0; sl < G::kSlices; ++sl)
            tma_prefetch_3d(&tmQ, sl * 64, e.kh * g, e.n0 + e.row0);
        }
      }
      if (__shfl_sync(0xffffffffu, it.x, 0) < 0) break;
    }
  } else if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t k_issued = 0, k_par = 0, v_issued = 0, v_par = 0, q_issued = 0, q_par = 0;
      int Tk = 0, Tv = 0, v = 0;  // K and V tiles issued so far, items processed so far
      bool ok = true;
      for (int u = 0; ok; ++u) {
        const int slot = u & 1;
        if (!mbar_wait(item_full + slot, (u >> 1) & 1, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        if (ring[slot].it.x < 0) break;
        const ItemGeo e = ring[slot].e;
        // the query block: rb rows x g heads x d of the group, once the last
        // QK^T of the previous item has read the old one
        if (v >= 1 && !mbar_wait(q_free, (v - 1) & 1, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        if (v == 0 && a.hold_first) {
          // test hook: the first query block never lands
        } else {
          mbar_arrive_expect_tx(q_full, uint32_t(G::kSlices) * 64 * 2 * g * rb);
#pragma unroll
          for (int sl = 0; sl < G::kSlices; ++sl)
            tma_load_3d(smem + sl * (kBV * 128), &tmQ, q_full, sl * 64, e.kh * g, e.n0 + e.row0,
                        pol);
          q_issued = 1;
          q_par = v & 1;
        }
        // K_j and V_j are issued as soon as their slots drain, whichever first
        int jk = 0, jv = 0;
        IdleClock clk;
        while (jv < e.ntiles) {
          bool progressed = false;
          if (jk < e.ntiles) {
            const int T = Tk + jk;
            const int s = T % kStages;
            const uint32_t ph = (T / kStages) & 1;
            if (mbar_test(k_empty + s, ph ^ 1u)) {
              uint8_t* ks = smem + G::kOffK + s * 2 * G::kKVBytes;
              mbar_arrive_expect_tx(k_full + s, G::kKVBytes);
              const bool pre = jk < e.npt;
              const CUtensorMap* mk = pre ? &tmK : &tmKc;
              const int key = pre ? e.p0 + e.k_begin + jk * kBN : e.f_begin + (jk - e.npt) * kBN;
#pragma unroll
              for (int sl = 0; sl < G::kSlices; ++sl)
                tma_load_3d(ks + sl * (kBN * 128), mk, k_full + s, sl * 64, e.kh, key, pol);
              k_issued |= 1u << s;
              k_par = (k_par & ~(1u << s)) | (ph << s);
              ++jk;
              progressed = true;
            }
          }
          if (jv < jk) {
            const int T = Tv + jv;
            const int s = T % kStages;
            const uint32_t ph = (T / kStages) & 1;
            if (mbar_test(v_empty + s, ph ^ 1u)) {
              uint8_t* vs = smem + G::kOffK + s * 2 * G::kKVBytes + G::kKVBytes;
              mbar_arrive_expect_tx(v_full + s, G::kKVBytes);
              const bool pre = jv < e.npt;
              const CUtensorMap* mv = pre ? &tmV : &tmVc;
              const int key = pre ? e.p0 + e.k_begin + jv * kBN : e.f_begin + (jv - e.npt) * kBN;
#pragma unroll
              for (int sl = 0; sl < G::kSlices; ++sl)
                tma_load_3d(vs + sl * (kBN * 128), mv, v_full + s, sl * 64, e.kh, key, pol);
              v_issued |= 1u << s;
              v_par = (v_par & ~(1u << s)) | (ph << s);
              ++jv;
              progressed = true;
            }
          }
          if (clk.expired(progressed, abort_flag, a.wait_ns)) {
            ok = false;
            break;
          }
        }
        if (!ok) break;
        mbar_arrive(item_empty + slot);
        Tk += e.ntiles;
        Tv += e.ntiles;
        ++v;
      }
      if (!ok) {
        *abort_flag = 1;
        flag(a.status, JET_ERR_TIMEOUT);
        // let every copy already issued land before the CTA can exit
        if (q_issued) mbar_wait(q_full, q_par, kDrainNs, nullptr);
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
      bool ok = mbar_wait(qz_done, 0, a.wait_ns, abort_flag);
      int T = 0, v = 0;  // tiles and items processed so far
      for (int u = 0; ok; ++u) {
        const int slot = u & 1;
        if (!mbar_wait(item_full + slot, (u >> 1) & 1, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        if (ring[slot].it.x < 0) break;
        const ItemGeo e = ring[slot].e;
        if (!mbar_wait(q_full, v & 1, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // issue S_j = Q K_j^T and O += P_j V_j in whichever order their inputs
        // become ready; S_j always precedes P_j V_j
        int js = 0, jo = 0;
        IdleClock clk;
        while (ok && jo < e.ntiles) {
          bool progressed = false;
          if (js < e.ntiles) {
            const int Tj = T + js;
            const int s = Tj % kStages, b = Tj & 1;
            if (mbar_test(k_full + s, (Tj / kStages) & 1) &&
                mbar_test(s_free + b, ((Tj >> 1) & 1) ^ 1u)) {
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
              if (js == e.ntiles - 1) mma_commit(q_free);  // the query block may be replaced
              ++js;
              progressed = true;
            }
          }
          if (jo < js) {
            const int Tj = T + jo;
            const int s = Tj % kStages, b = Tj & 1;
            // the item's first P V overwrites O: the previous item's O must be out
            const bool o_ready = jo > 0 || v == 0 || mbar_test(o_free, (v - 1) & 1);
            if (o_ready && mbar_test(p_full + b, (Tj >> 1) & 1) &&
                mbar_test(v_full + s, (Tj / kStages) & 1)) {
              tc_fence_after();
              // P_j from TMEM (8 columns = 16 keys per instruction), V_j from shared memory
              const uint32_t pt = tmem + G::kPCol + uint32_t(b) * (kBN / 2);
              const uint32_t vs = smem_u32(smem + G::kOffK + s * 2 * G::kKVBytes + G::kKVBytes);
#pragma unroll
              for (int k = 0; k < kBN / 16; ++k)
                mma_f16_ta(tmem + G::kOCol, pt + uint32_t(8 * k),
                           desc_mn_sw128(vs + k * 16 * 128, kBN * 128), id_o, (jo | k) != 0);
              mma_commit(p_free + b);
              mma_commit(v_empty + s);
              ++jo;
              progressed = true;
            }
          }
          if (clk.expired(progressed, abort_flag, a.wait_ns)) ok = false;
        }
        if (!ok) break;
        mbar_arrive(item_empty + slot);
        T += e.ntiles;
        ++v;
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
    // the output is transposed through this warp's own 4 KB of the output
    // stage so that every global store covers whole 64- or 128-byte pieces of
    // one vector's output
    uint4* stage = reinterpret_cast<uint4*>(smem + G::kOffStage + q4 * 32 * 128);
    // the query blocks arrive by TMA (rows [0, rb g)); zero the rows past them
    // once so that no stale shared memory enters the MMA
    if (i >= rb * g) {
#pragma unroll
      for (int c = 0; c < DH / 8; ++c)
        *reinterpret_cast<uint4*>(smem + (c >> 3) * (kBV * 128) + sw128(i, c & 7)) =
            make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(qz_done);

    bool ok = true;
    int T = 0;
    for (int u = 0; ok; ++u) {
      const int slot = u & 1;
      if (!warp_mbar_wait(item_full + slot, (u >> 1) & 1, a.wait_ns, abort_flag)) {
        ok = false;
        break;
      }
      if (ring[slot].it.x < 0) break;
      const ItemGeo e = ring[slot].e;
      const bool valid = i < e.nv;
      int fa = 1, fb = 0;  // fed-token indices this vector may see (none: shared row)
      // prefill: the last key this vector's position may see (causal)
      const int kcap = a.prefill ? (e.vbase + i) / g : (1 << 30);
      if (valid && !a.prefill) {
        const int gv = e.vbase + i;
        const int n = e.n0 + gv / g;
        const int c = a.row_cand[n];
        if (c >= 0 && c < a.C) {
          fa = a.cand_row_offset[c] - e.r - 1;  // y_{c,1}
          fb = n - e.r - 1;                     // the row's own fed token, inclusive
        }
      }
      float m_used = -INFINITY, l = 0.f;
      for (int j = 0; j < e.ntiles; ++j) {
        const int Tj = T + j;
        const int b = Tj & 1;
        if (!warp_mbar_wait(s_full + b, (Tj >> 1) & 1, a.wait_ns, abort_flag)) {
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
        if (j < e.npt) {
          khi = min(kBN, e.k_end - (e.k_begin + j * kBN));
          khi = min(khi, kcap + 1 - (e.k_begin + j * kBN));  // prefill: keys <= own position
        } else {
          const int f0 = e.f_begin + (j - e.npt) * kBN;
          klo = max(0, fa - f0);
          khi = min(kBN, fb - f0 + 1);
        }
        // the row's tile maximum through eight independent chains (one warp per
        // scheduler runs this: a single 64-long chain would be pure latency)
        float mq[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) mq[q] = -INFINITY;
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          sv[c] = (c >= klo && c < khi) ? sv[c] * a.scale_log2 : -INFINITY;
          mq[c & 7] = fmaxf(mq[c & 7], sv[c]);
        }
        const float mt = fmaxf(fmaxf(fmaxf(mq[0], mq[1]), fmaxf(mq[2], mq[3])),
                               fmaxf(fmaxf(mq[4], mq[5]), fmaxf(mq[6], mq[7])));
        // P buffer b was last read by the P V of tile Tj - 2
        if (Tj >= 2 && !warp_mbar_wait(p_free + b, ((Tj - 2) >> 1) & 1, a.wait_ns, abort_flag)) {
          ok = false;
          break;
        }
        if (mt > m_used + kRescaleLog2) {
          const float m_new = mt;
          if (j >= 1) {
            // O holds this item's P V so far: wait for the last one, rescale in TMEM
            if (!warp_mbar_wait(p_free + ((Tj - 1) & 1), ((Tj - 1) >> 1) & 1, a.wait_ns,
                                abort_flag)) {
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
        // P = 2^(s - m_used) as bf16 pairs into this row's TMEM lane (the P V
        // MMA's A operand); the row sum uses the rounded values, which are what
        // the tensor core multiplies
        uint32_t pw[kBN / 2];
        float ps[8];  // one partial sum per 8 keys, added as a tree
#pragma unroll
        for (int cc = 0; cc < 8; ++cc) {
          ps[cc] = 0.f;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float x0 = ex2(sv[cc * 8 + 2 * q] - m_used);
            const float x1 = ex2(sv[cc * 8 + 2 * q + 1] - m_used);
            pw[cc * 4 + q] = pack_bf16(x0, x1);
            const __nv_bfloat162 hb = *reinterpret_cast<const __nv_bfloat162*>(&pw[cc * 4 + q]);
            ps[cc] += __bfloat162float(hb.x) + __bfloat162float(hb.y);
          }
        }
        tmem_st_32cols_u32(tmem + lane_off + G::kPCol + uint32_t(b) * (kBN / 2), pw);
        l += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(p_full + b);
      }
      if (!ok) break;
      // wait for the item's last P V, then write its output (or its partial)
      const int Tl = T + e.ntiles - 1;
      if (!warp_mbar_wait(p_free + (Tl & 1), (Tl >> 1) & 1, a.wait_ns, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const bool direct = e.splits_r == 1;  // the whole row in this item: final output
      if (valid) {
        const int gv = e.vbase + i;
        const int n = e.n0 + gv / g, h = e.kh * g + gv % g;
        if (!direct) a.ml_part[(size_t(e.split) * a.N + n) * a.Hq + h] = make_float2(m_used, l);
      }
      // the destination of the vectors this lane stores: vector 4 s + lane / 8
      // (f32 partial, 8 lanes x 16 bytes each) or 8 s + lane / 4 (bf16 output,
      // 4 lanes x 16 bytes each); element offsets, -1 past the block's vectors
      long long dst[8];
#pragma unroll
      for (int s = 0; s < 8; ++s) {
        const int iv = direct ? 8 * s + (lane >> 2) : 4 * s + (lane >> 3);
        const int gi = q4 * 32 + iv;
        dst[s] = -1;
        if ((!direct || s < 4) && gi < e.nv) {
          const int gv = e.vbase + gi;
          const int n = e.n0 + gv / g, h = e.kh * g + gv % g;
          dst[s] = direct ? (long long)(size_t(n) * a.Hq + h) * DH
                          : (long long)((size_t(e.split) * a.N + n) * a.Hq + h) * DH;
        }
      }
      const float inv = l > 0.f ? 1.f / l : 0.f;
      // 64 columns of O per TMEM round trip, written as two 32-column pieces
#pragma unroll 1
      for (int c0 = 0; c0 < DH; c0 += 64) {
        float ovp[2][32];
        tmem_ld_32cols(tmem + lane_off + G::kOCol + c0, ovp[0]);
        tmem_ld_32cols(tmem + lane_off + G::kOCol + c0 + 32, ovp[1]);
        tmem_wait_ld();
#pragma unroll
        for (int hp = 0; hp < 2; ++hp) {
          const float* ov = ovp[hp];
          const int cc0 = c0 + 32 * hp;
          if (direct) {
            // 32 bf16 = four 16-byte pieces per vector; two vectors per 128-byte
            // row of the stage, pieces rotated so that 8 lanes hit 8 bank groups
#pragma unroll
            for (int q = 0; q < 4; ++q)
              stage[(lane >> 1) * 8 + (lane & 1) * 4 + (q ^ ((lane >> 1) & 3))] =
                  make_uint4(pack_bf16(ov[8 * q] * inv, ov[8 * q + 1] * inv),
                             pack_bf16(ov[8 * q + 2] * inv, ov[8 * q + 3] * inv),
                             pack_bf16(ov[8 * q + 4] * inv, ov[8 * q + 5] * inv),
                             pack_bf16(ov[8 * q + 6] * inv, ov[8 * q + 7] * inv));
            __syncwarp();
#pragma unroll
            for (int s = 0; s < 4; ++s) {
              const int iv = 8 * s + (lane >> 2), c = lane & 3;
              const uint4 val = stage[(iv >> 1) * 8 + (iv & 1) * 4 + (c ^ ((iv >> 1) & 3))];
              if (dst[s] >= 0) *reinterpret_cast<uint4*>(a.o + dst[s] + cc0 + c * 8) = val;
            }
          } else {
            // 32 f32 = eight 16-byte pieces per vector, one vector per 128-byte
            // row of the stage, pieces rotated by the row
#pragma unroll
            for (int q = 0; q < 8; ++q)
              stage[lane * 8 + (q ^ (lane & 7))] =
                  make_uint4(__float_as_uint(ov[4 * q]), __float_as_uint(ov[4 * q + 1]),
                             __float_as_uint(ov[4 * q + 2]), __float_as_uint(ov[4 * q + 3]));
            __syncwarp();
#pragma unroll
            for (int s = 0; s < 8; ++s) {
              const int iv = 4 * s + (lane >> 3), c = lane & 7;
              const uint4 val = stage[iv * 8 + (c ^ (iv & 7))];
              if (dst[s] >= 0) *reinterpret_cast<uint4*>(a.o_part + dst[s] + cc0 + c * 4) = val;
            }
          }
          __syncwarp();
        }
      }
      // O may be overwritten by the next item's first P V; the ring slot is free
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(o_free);
        mbar_arrive(item_empty + slot);
      }
      T += e.ntiles;
    }
    if (!ok) {
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
  pdl_begin();
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
  int per = 0;
  const int splits_r = req_splits(P, chunk, &per);
  if (splits_r <= 1) return;
  constexpr int PER = DH / 32;
  float acc[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) acc[i] = 0.f;
  float m = -INFINITY, l = 0.f;
  // four chunks' partials at a time, every load issued before the first is
  // used (the chunks are combined in order)
  constexpr int kGroup = 4;
  for (int s0 = 0; s0 < splits_r; s0 += kGroup) {
    float2 ml[kGroup];
    float v[kGroup][PER];
#pragma unroll
    for (int q = 0; q < kGroup; ++q) {
      ml[q] = make_float2(-INFINITY, 0.f);
      if (s0 + q < splits_r) {
        const size_t base = (size_t(s0 + q) * N + n) * Hq + h;
        ml[q] = ml_part[base];
#pragma unroll
        for (int i = 0; i < PER; ++i) v[q][i] = o_part[base * DH + lane + 32 * i];
      }
    }
#pragma unroll
    for (int q = 0; q < kGroup; ++q) {
      if (!(ml[q].y > 0.f)) continue;
      const float mn = fmaxf(m, ml[q].x);
      const float fa = exp2f(m - mn), fb = exp2f(ml[q].x - mn);
#pragma unroll
      for (int i = 0; i < PER; ++i) acc[i] = acc[i] * fa + v[q][i] * fb;
      l = l * fa + ml[q].y * fb;
      m = mn;
    }
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
  a.wait_ns = wait_budget_ns();
  a.hold_first = test_stall();
  a.prefix_offset = lay.prefix_offset;
  a.row_offset = lay.row_offset;
  a.req_order = lay.req_order;
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
  a.g = g;
  a.rb = kBV / g;
  a.has_cand = F > 0;
  a.scale_log2 = 1.4426950408889634f / sqrtf(float(DH));
  // the work list follows the (m, l) partials in the workspace
  const size_t vecs = size_t(plan.splits) * n.N * d.Hq;
  uintptr_t ctrl = reinterpret_cast<uintptr_t>(ml_part + vecs);
  ctrl = (ctrl + 15) & ~uintptr_t(15);
  a.item_next = reinterpret_cast<int*>(ctrl);
  a.item_count = a.item_next + 1;
  a.items = reinterpret_cast<int4*>(ctrl + 16);
  a.splits = plan.splits;
  a.n_all = (long long)n.R * d.Hkv * plan.qgroups * plan.splits;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return cudaErrorInvalidValue;
  const int grid = int(std::max<long long>(1, std::min<long long>(sms, a.n_all)));
  // longest-first dynamic order pays for its extra launch only when items are
  // long and uneven (chunks of 16 key tiles or more); a grid that covers every
  // slot takes one slot per CTA and needs no shared counter
  a.sorted = plan.chunk >= 16 * kBN;
  a.static_only = !a.sorted && a.n_all <= grid;
  cudaError_t e = cudaSuccess;
  if (a.sorted)
    e = launch_pdl(attend_items_kernel, dim3(1), dim3(1024), 0, st, a, plan.qgroups, plan.splits);
  else if (!a.static_only)
    e = launch_pdl(attend_reset_kernel, dim3(1), dim3(128), 0, st, a.item_next, a.prefix_offset,
                   a.row_offset, a.req_order, a.row_cand, a.cand_row_offset, a.R, a.N, a.C);
  if (e != cudaSuccess) return e;
  const size_t smem = Geo<DH>::kBytes + 1024;
  e = cudaFuncSetAttribute(attend_prefix_tc_kernel<DH>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  e = launch_pdl(attend_prefix_tc_kernel<DH>, dim3(grid), dim3(kThreads), smem, st, tmQ, tmK, tmV,
                 tmKc, tmVc, a);
  if (e != cudaSuccess || plan.splits <= 1) return e;
  const long long warps = (long long)n.N * d.Hq;
  return launch_pdl(attend_combine_kernel<DH>, dim3(unsigned((warps + 7) / 8)), dim3(256), 0, st,
                    lay.prefix_offset, lay.row_req, n.N, n.R, d.Hq, plan.chunk, o_part, ml_part,
                    static_cast<__nv_bfloat16*>(o), status);
}

// Prefill: causal self-attention over every request's prefix with the same
// persistent kernel. Items are (request, kv head, block of 128/g positions):
// a block reads the keys up to its last position, a row masks the keys past
// its own; no chunking (the blocks already give one item per 128 / g
// positions), so the output is written directly. Longest items first.
template <int DH>
cudaError_t launch_prefill_dh(const jet_layout& lay, const jet_dims& d, const void* q,
                              const void* k, const void* v, void* o, void* ws, int* status,
                              cudaStream_t st) {
  const jet_sizes& n = lay.n;
  const int g = d.Hq / d.Hkv;
  if (g > kBV) return cudaErrorInvalidValue;
  CUtensorMap tmQ, tmK, tmV;
  if (!encode_3d(&tmQ, q, n.total_prefix, d.Hq, DH, g, kBV / g) ||
      !encode_3d(&tmK, k, n.total_prefix, d.Hkv, DH, 1, kBN) ||
      !encode_3d(&tmV, v, n.total_prefix, d.Hkv, DH, 1, kBN))
    return cudaErrorInvalidValue;
  AttArgs a{};
  a.wait_ns = wait_budget_ns();
  a.hold_first = test_stall();
  a.prefix_offset = lay.prefix_offset;
  a.row_offset = lay.row_offset;
  a.req_order = lay.req_order;
  a.row_cand = lay.row_cand;
  a.cand_row_offset = lay.cand_row_offset;
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.o = static_cast<__nv_bfloat16*>(o);
  a.status = status;
  a.R = n.R;
  a.N = n.total_prefix;
  a.C = 0;
  a.total_prefix = n.total_prefix;
  a.Hq = d.Hq;
  a.Hkv = d.Hkv;
  a.chunk = 1 << 30;
  a.g = g;
  a.rb = kBV / g;
  a.has_cand = 0;
  a.prefill = 1;
  a.scale_log2 = 1.4426950408889634f / sqrtf(float(DH));
  const int qgroups = (n.max_prefix + a.rb - 1) / a.rb;
  uintptr_t ctrl = (reinterpret_cast<uintptr_t>(ws) + 15) & ~uintptr_t(15);
  a.item_next = reinterpret_cast<int*>(ctrl);
  a.item_count = a.item_next + 1;
  a.items = reinterpret_cast<int4*>(ctrl + 16);
  a.splits = 1;
  a.n_all = (long long)n.R * d.Hkv * qgroups;
  a.sorted = 1;
  cudaError_t e =
      launch_pdl(attend_items_kernel, dim3(1), dim3(1024), 0, st, a, qgroups, 1);
  if (e != cudaSuccess) return e;
  const size_t smem = Geo<DH>::kBytes + 1024;
  e = cudaFuncSetAttribute(attend_prefix_tc_kernel<DH>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
    return cudaErrorInvalidValue;
  const int grid = int(std::max<long long>(1, std::min<long long>(sms, a.n_all)));
  return launch_pdl(attend_prefix_tc_kernel<DH>, dim3(grid), dim3(kThreads), smem, st, tmQ, tmK,
                    tmV, tmK, tmV, a);
}

}  // namespace

int attn_tc_block() { return kBV; }

size_t prefill_workspace_bytes(const jet_sizes& n, const jet_dims& d) {
  if (d.Hkv < 1 || d.Hq < d.Hkv || d.Hq % d.Hkv != 0) return 0;
  const int g = d.Hq / d.Hkv;
  if (g > kBV) return 0;
  const int rb = kBV / g;
  const long long qgroups = (n.max_prefix + rb - 1) / rb;
  return 32 + 16 * size_t(n.R) * d.Hkv * qgroups;
}

cudaError_t launch_prefill_tc(const jet_layout& lay, const jet_dims& d, const void* q,
                              const void* k, const void* v, void* o, void* ws, int* status,
                              cudaStream_t st) {
  if (d.d == 64) return launch_prefill_dh<64>(lay, d, q, k, v, o, ws, status, st);
  if (d.d == 128) return launch_prefill_dh<128>(lay, d, q, k, v, o, ws, status, st);
  if (d.d == 256) return launch_prefill_dh<256>(lay, d, q, k, v, o, ws, status, st);
  return cudaErrorInvalidValue;
}

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
