// Candidate scoring for callers that cannot allocate device memory.
//
// jet_score_candidates needs scratch memory (per-tile log-sum-exp partials,
// gathered target logits, per-row log-sum-exp) that its caller allocates and
// passes in. Some callers cannot do that: a host application that owns every
// device allocation and hands its plug-ins only the tensors they work on, or a
// serving loop that must not call cudaMalloc once it runs (cudaMalloc can
// synchronise the device, and it can fail under memory pressure in the middle
// of a request). jet_score_candidates_noalloc serves them with a fixed scratch
// array that lives in the library itself: a file-scope __device__ array,
// created when the library's module loads on a device and held by every GPU
// that loads the library until the process exits.
#include <mutex>

#include "jet.h"
#include "jet_internal.h"

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;  // 16 MiB

__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array on the current device. In host code
// the array's name is only a host-side stand-in, so the address is looked up
// with cudaGetSymbolAddress once per device, with that device current.
jet_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return JET_ERR_CUDA;
  static std::mutex mu;
  static void* addr[64] = {};
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return JET_ERR_CUDA;
    addr[dev] = p;
  }
  *out = addr[dev];
  return JET_OK;
}

}  // namespace

extern "C" jet_status jet_score_candidates_noalloc(const jet_layout* lay, const jet_dims* dims,
                                                   const void* hidden, const void* w_lm,
                                                   float* tok_logprob, float* cand_score,
                                                   void* stream) {
  if (!lay) return JET_ERR_ARG;
  if (lay->n.R > 0 && lay->n.N > 0 && lay->n.V > 0 &&
      jet::score_plan(lay->n).bytes > kNoAllocScratchBytes)
    return JET_ERR_CAPACITY;  // this batch needs more scratch than the fixed array holds
  void* scratch = nullptr;
  if (lay->n.R > 0) {
    const jet_status s = scratch_address(&scratch);
    if (s != JET_OK) return s;
  }
  // Every scratch element the call reads is written earlier in the same call,
  // so nothing has to be cleared between calls.
  return jet_score_candidates(lay, dims, hidden, w_lm, tok_logprob, cand_score, scratch,
                              kNoAllocScratchBytes, stream);
}
