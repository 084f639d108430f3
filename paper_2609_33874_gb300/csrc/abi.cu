// The C entry points of libjet: argument validation, workspace plans and
// stream-ordered launches. No entry point allocates memory, synchronises a
// stream (except jet_device_status) or launches anything after a failed
// check.
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <mutex>

#include "jet.h"

#include "jet_internal.h"

namespace jet {

// Per-device status word written by kernels that meet an out-of-range layout
// index or give up a bounded wait.
__device__ int g_status_word;

namespace {
constexpr uint64_t kDefaultWaitNs = 2000000000ull;
std::atomic<uint64_t> g_wait_ns{kDefaultWaitNs};
std::atomic<uint64_t> g_launches{0};
std::atomic<int> g_test_stall{0};
}  // namespace

uint64_t wait_budget_ns() { return g_wait_ns.load(std::memory_order_relaxed); }

int test_stall() { return g_test_stall.load(std::memory_order_relaxed); }

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int* device_status_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  static std::mutex mu;
  static int* ptrs[64] = {};
  std::lock_guard<std::mutex> lock(mu);
  if (!ptrs[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    ptrs[dev] = static_cast<int*>(p);
  }
  return ptrs[dev];
}

// bf16 runs on the tensor cores; float32 keeps float32 FMA (tf32 tensor-core
// inputs would round it)
cudaError_t launch_lmhead(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                          const void* hidden, const void* w_lm, void* ws, int* status,
                          cudaStream_t st) {
  if (d.dtype == JET_DTYPE_BF16)
    return launch_lmhead_tc(lay, d, plan, hidden, w_lm, ws, status, st);
  return launch_lmhead_simt(lay, d, plan, hidden, w_lm, ws, status, st);
}

}  // namespace jet

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// A device pointer argument: non-null and 16-byte aligned when it will be
// touched (count > 0).
jet_status check_ptr(const void* p, long long count) {
  if (count <= 0) return JET_OK;
  if (!p) return JET_ERR_ARG;
  if (!aligned16(p)) return JET_ERR_ALIGN;
  return JET_OK;
}

jet_status check_layout(const jet_layout* lay) {
  if (!lay) return JET_ERR_ARG;
  const jet_sizes& n = lay->n;
  if (n.R < 0 || n.C < 0 || n.N < 0 || n.T < 0 || n.V < 1) return JET_ERR_SHAPE;
  if (n.R == 0) return JET_OK;
  if (n.C < n.R || n.N < n.R || n.T < n.C || n.total_prefix < n.R || n.max_prefix < 1 ||
      n.max_prefix > n.total_prefix || n.min_cand < 1 || n.max_cand < n.min_cand ||
      n.max_rows < 1 || n.max_rows > n.N || n.max_len < 1 || n.N - n.R != n.T - n.C)
    return JET_ERR_SHAPE;
  const void* arrays[13] = {lay->prefix_offset, lay->cand_offset,    lay->row_offset,
                            lay->cand_row_offset, lay->tgt_offset,   lay->target_ids,
                            lay->tgt_row,       lay->row_req,        lay->row_cand,
                            lay->row_pos,       lay->row_tgt_offset, lay->row_tgt_index,
                            lay->req_order};
  for (const void* a : arrays)
    if (!a) return JET_ERR_ARG;
  return JET_OK;
}

jet_status check_dtype(const jet_dims* d) {
  if (!d) return JET_ERR_ARG;
  if (d->dtype != JET_DTYPE_F32 && d->dtype != JET_DTYPE_BF16) return JET_ERR_UNSUPPORTED;
  return JET_OK;
}

jet_status check_attn_dims(const jet_dims* d) {
  jet_status s = check_dtype(d);
  if (s) return s;
  if (d->Hq < 1 || d->Hkv < 1 || d->Hq % d->Hkv != 0) return JET_ERR_SHAPE;
  if (d->d != 64 && d->d != 128 && d->d != 256) return JET_ERR_UNSUPPORTED;
  return JET_OK;
}

jet_status check_lm_dims(const jet_dims* d) {
  jet_status s = check_dtype(d);
  if (s) return s;
  if (d->D < 8 || d->D % 8 != 0) return JET_ERR_SHAPE;
  if (d->max_sms < 0) return JET_ERR_ARG;
  return JET_OK;
}

jet_status check_fork_dims(const jet_dims* d) {
  jet_status s = check_dtype(d);
  if (s) return s;
  if (d->Hl < 1 || d->dk < 1 || d->dv < 1) return JET_ERR_SHAPE;
  if (d->dk != 128 || d->dv % 32 != 0) return JET_ERR_UNSUPPORTED;
  return JET_OK;
}

jet_status check_e4m3_dims(const jet_dims* d) {
  if (!d) return JET_ERR_ARG;
  if (d->dtype != JET_DTYPE_BF16) return JET_ERR_UNSUPPORTED;
  if (d->D < 16 || d->D % 16 != 0) return JET_ERR_SHAPE;
  if (d->max_sms < 0) return JET_ERR_ARG;
  return JET_OK;
}

// scratch of the e4m3 score path: the bf16 path's plan, then the hidden
// states' codes [N, D] and scales [N]
struct E4m3Plan {
  jet::ScorePlan score;
  size_t hq_off, hs_off, bytes;
};

E4m3Plan e4m3_plan(const jet_sizes& n, int D) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  E4m3Plan p{};
  p.score = jet::score_plan(n);
  p.hq_off = up(p.score.bytes);
  p.hs_off = p.hq_off + up(size_t(n.N) * size_t(D));
  p.bytes = p.hs_off + up(size_t(n.N) * sizeof(float));
  return p;
}

// scratch of the MXFP8 score path: the bf16 path's plan, then the hidden
// states' codes [N, D] and their scale factors (two 512-byte chunks per token
// tile and K slice)
struct MxPlan {
  jet::ScorePlan score;
  size_t hq_off, hsf_off, bytes;
  int Nt, n_tt;
};

MxPlan mx_plan(const jet_sizes& n, int D) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  MxPlan p{};
  p.score = jet::score_plan(n);
  jet::mx_token_tiling(n.N > 0 ? n.N : 1, &p.Nt, &p.n_tt);
  const size_t nkb = size_t(D + 127) / 128;
  p.hq_off = up(p.score.bytes);
  p.hsf_off = p.hq_off + up(size_t(n.N) * size_t(D));
  p.bytes = p.hsf_off + size_t(p.n_tt) * nkb * 2 * jet::kW4ScaleBytes;
  return p;
}

// bytes of the MXFP8 weight buffer: codes [V, D], then one 512-byte chunk of
// scale factors per (128-row tile, 128-element K slice)
size_t mx_weight_bytes(int64_t V, int64_t D) {
  const size_t codes = (size_t(V) * size_t(D) + 255) & ~size_t(255);
  return codes + size_t((V + 127) / 128) * size_t((D + 127) / 128) * jet::kW4ScaleBytes;
}

jet_status cuda_status(cudaError_t e) { return e == cudaSuccess ? JET_OK : JET_ERR_CUDA; }

#define JET_TRY(expr)            \
  do {                           \
    jet_status s_ = (expr);      \
    if (s_ != JET_OK) return s_; \
  } while (0)

}  // namespace

extern "C" int32_t jet_abi_version(void) { return JET_ABI_VERSION; }

extern "C" const char* jet_status_string(jet_status s) {
  switch (s) {
    case JET_OK: return "ok";
    case JET_ERR_ARG: return "invalid argument (null pointer or bad scalar)";
    case JET_ERR_SHAPE: return "inconsistent sizes";
    case JET_ERR_RANGE: return "token id outside [0, V)";
    case JET_ERR_ALIGN: return "device pointer not 16-byte aligned";
    case JET_ERR_WORKSPACE: return "workspace missing or too small";
    case JET_ERR_CAPACITY: return "size beyond kernel capacity";
    case JET_ERR_UNSUPPORTED: return "unsupported dtype or dimension";
    case JET_ERR_CUDA: return "CUDA runtime error";
    case JET_ERR_TIMEOUT: return "bounded device wait gave up";
    case JET_ERR_DEVICE: return "kernel met an out-of-range layout index";
    default: return "unknown status";
  }
}

extern "C" size_t jet_workspace_bytes(const jet_sizes* n, const jet_dims* d) {
  if (!n || !d || n->R < 0 || n->N < 0 || n->V < 1) return 0;
  size_t a = 0, b = 0;
  if (d->Hq > 0 && d->Hkv > 0 && d->Hq % d->Hkv == 0 && d->d > 0) a = jet::attn_plan(*n, *d).bytes;
  b = jet::score_plan(*n).bytes;
  return a > b ? a : b;
}

extern "C" jet_status jet_prefix_attend(const jet_layout* lay, const jet_dims* dims, const void* q,
                                        const void* k_pre, const void* v_pre, const void* k_cand,
                                        const void* v_cand, void* o, void* ws, size_t ws_bytes,
                                        void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_attn_dims(dims));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  if ((long long)n.R * dims->Hkv > 65535) return JET_ERR_CAPACITY;
  const long long F = n.N - n.R;
  JET_TRY(check_ptr(q, n.N));
  JET_TRY(check_ptr(k_pre, n.total_prefix));
  JET_TRY(check_ptr(v_pre, n.total_prefix));
  JET_TRY(check_ptr(k_cand, F));
  JET_TRY(check_ptr(v_cand, F));
  JET_TRY(check_ptr(o, n.N));
  const jet::AttnPlan plan = jet::attn_plan(n, *dims);
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  return cuda_status(jet::launch_prefix_attend(*lay, *dims, plan, q, k_pre, v_pre, k_cand, v_cand, o,
                                               ws, jet::device_status_ptr(),
                                               static_cast<cudaStream_t>(stream)));
}

extern "C" size_t jet_prefill_workspace_bytes(const jet_sizes* n, const jet_dims* d) {
  if (!n || !d || n->R < 0) return 0;
  return jet::prefill_workspace_bytes(*n, *d);
}

extern "C" jet_status jet_prefill_attend(const jet_layout* lay, const jet_dims* dims,
                                         const void* q, const void* k, const void* v, void* o,
                                         void* ws, size_t ws_bytes, void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_attn_dims(dims));
  if (dims->dtype != JET_DTYPE_BF16) return JET_ERR_UNSUPPORTED;
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  const size_t need = jet::prefill_workspace_bytes(n, *dims);
  if (need == 0) return JET_ERR_SHAPE;
  if ((need - 32) / 16 > size_t(INT32_MAX)) return JET_ERR_CAPACITY;  // items a counter indexes
  JET_TRY(check_ptr(q, n.total_prefix));
  JET_TRY(check_ptr(k, n.total_prefix));
  JET_TRY(check_ptr(v, n.total_prefix));
  JET_TRY(check_ptr(o, n.total_prefix));
  if (!ws || ws_bytes < need) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  return cuda_status(jet::launch_prefill_tc(*lay, *dims, q, k, v, o, ws, jet::device_status_ptr(),
                                            static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_prefill_state(const jet_layout* lay, const jet_dims* dims, int32_t rule,
                                        const float* s_init, const void* q, const void* k,
                                        const void* v, const float* alpha, const float* beta,
                                        void* o, float* s_out, void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_fork_dims(dims));
  if (rule != JET_RECUR_DELTA && rule != JET_RECUR_GLA) return JET_ERR_ARG;
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  if (n.R > 65535 || dims->Hl > 65535) return JET_ERR_CAPACITY;
  if (s_init && !aligned16(s_init)) return JET_ERR_ALIGN;
  JET_TRY(check_ptr(q, n.total_prefix));
  JET_TRY(check_ptr(k, n.total_prefix));
  JET_TRY(check_ptr(v, n.total_prefix));
  JET_TRY(check_ptr(alpha, n.total_prefix));
  JET_TRY(check_ptr(beta, n.total_prefix));
  JET_TRY(check_ptr(o, n.total_prefix));
  JET_TRY(check_ptr(s_out, n.R));
  return cuda_status(jet::launch_prefill_state(*lay, *dims, rule, s_init, q, k, v, alpha, beta, o,
                                               s_out, jet::device_status_ptr(),
                                               static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_fork_state_rule(const jet_layout* lay, const jet_dims* dims,
                                          int32_t rule, const float* s_prefix, const void* q,
                                          const void* k, const void* v, const float* alpha,
                                          const float* beta, void* o, float* s_fork,
                                          void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_fork_dims(dims));
  if (rule != JET_RECUR_DELTA && rule != JET_RECUR_GLA) return JET_ERR_ARG;
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  if (n.R > 65535 || dims->Hl > 65535) return JET_ERR_CAPACITY;
  const long long F = n.N - n.R;
  JET_TRY(check_ptr(s_prefix, n.R));
  JET_TRY(check_ptr(q, F));
  JET_TRY(check_ptr(k, F));
  JET_TRY(check_ptr(v, F));
  JET_TRY(check_ptr(alpha, F));
  JET_TRY(check_ptr(beta, F));
  JET_TRY(check_ptr(o, F));
  if (s_fork && !aligned16(s_fork)) return JET_ERR_ALIGN;
  return cuda_status(jet::launch_fork_state(*lay, *dims, rule, s_prefix, q, k, v, alpha, beta, o,
                                            s_fork, jet::device_status_ptr(),
                                            static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_fork_state(const jet_layout* lay, const jet_dims* dims,
                                     const float* s_prefix, const void* q, const void* k,
                                     const void* v, const float* alpha, const float* beta, void* o,
                                     float* s_fork, void* stream) {
  return jet_fork_state_rule(lay, dims, JET_RECUR_DELTA, s_prefix, q, k, v, alpha, beta, o,
                             s_fork, stream);
}

extern "C" jet_status jet_score_candidates(const jet_layout* lay, const jet_dims* dims,
                                           const void* hidden, const void* w_lm,
                                           float* tok_logprob, float* cand_score, void* ws,
                                           size_t ws_bytes, void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_lm_dims(dims));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  const jet::ScorePlan plan = jet::score_plan(n);
  if (plan.vtiles > 65535) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(hidden, n.N));
  JET_TRY(check_ptr(w_lm, n.V));
  JET_TRY(check_ptr(tok_logprob, n.T));
  JET_TRY(check_ptr(cand_score, n.C));
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  int* status = jet::device_status_ptr();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  JET_TRY(cuda_status(jet::launch_lmhead(*lay, *dims, plan, hidden, w_lm, ws, status, st)));
  return cuda_status(jet::launch_score_finish(*lay, plan, ws, tok_logprob, cand_score, status, st));
}

extern "C" jet_status jet_quantize_rows_e4m3(const void* x, int32_t rows, int32_t D, uint8_t* q,
                                             float* scale, void* stream) {
  if (rows < 0) return JET_ERR_ARG;
  if (D < 16 || D % 16 != 0) return JET_ERR_SHAPE;
  if (rows == 0) return JET_OK;
  JET_TRY(check_ptr(x, rows));
  JET_TRY(check_ptr(q, rows));
  JET_TRY(check_ptr(scale, rows));
  return cuda_status(jet::launch_quantize_e4m3(x, rows, D, q, scale,
                                               static_cast<cudaStream_t>(stream)));
}

extern "C" size_t jet_workspace_bytes_e4m3(const jet_sizes* n, const jet_dims* d) {
  if (!n || !d || n->R < 0 || n->N < 0 || n->V < 1 || d->D < 16) return 0;
  size_t a = 0;
  if (d->Hq > 0 && d->Hkv > 0 && d->Hq % d->Hkv == 0 && d->d > 0) a = jet::attn_plan(*n, *d).bytes;
  const size_t b = e4m3_plan(*n, d->D).bytes;
  return a > b ? a : b;
}

extern "C" jet_status jet_score_candidates_e4m3(const jet_layout* lay, const jet_dims* dims,
                                                const void* hidden, const uint8_t* w_q,
                                                const float* w_scale, float* tok_logprob,
                                                float* cand_score, void* ws, size_t ws_bytes,
                                                void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_e4m3_dims(dims));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  const E4m3Plan plan = e4m3_plan(n, dims->D);
  if (plan.score.vtiles > 65535) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(hidden, n.N));
  JET_TRY(check_ptr(w_q, n.V));
  JET_TRY(check_ptr(w_scale, n.V));
  JET_TRY(check_ptr(tok_logprob, n.T));
  JET_TRY(check_ptr(cand_score, n.C));
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  int* status = jet::device_status_ptr();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* h_q = static_cast<uint8_t*>(ws) + plan.hq_off;
  float* h_scale = reinterpret_cast<float*>(static_cast<char*>(ws) + plan.hs_off);
  JET_TRY(cuda_status(jet::launch_quantize_e4m3(hidden, n.N, dims->D, h_q, h_scale, st)));
  JET_TRY(cuda_status(jet::launch_lmhead_e4m3(*lay, *dims, plan.score, h_q, h_scale, w_q, w_scale,
                                              ws, status, st)));
  return cuda_status(
      jet::launch_score_finish(*lay, plan.score, ws, tok_logprob, cand_score, status, st));
}

extern "C" size_t jet_w4_bytes(int64_t V, int64_t D) {
  if (V < 1 || D < 16 || D % 16 != 0 || V > (int64_t(1) << 31) || D > (int64_t(1) << 31))
    return 0;
  return size_t((V + jet::kVocabTile - 1) / jet::kVocabTile) * size_t((D + 127) / 128) *
         size_t(jet::kW4TileBytes);
}

extern "C" jet_status jet_quantize_w4(const void* w, int64_t V, int64_t D, uint8_t* w4,
                                      float* scale, void* stream) {
  if (V < 1) return JET_ERR_ARG;
  if (D < 16 || D % 16 != 0) return JET_ERR_SHAPE;
  if (V > (int64_t(1) << 30) || D > (int64_t(1) << 20)) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(w, V));
  JET_TRY(check_ptr(w4, V));
  JET_TRY(check_ptr(scale, V));
  return cuda_status(jet::launch_quantize_w4(w, int(V), int(D), w4, scale,
                                             static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_score_candidates_w4(const jet_layout* lay, const jet_dims* dims,
                                              const void* hidden, const uint8_t* w4,
                                              const float* w_scale, float* tok_logprob,
                                              float* cand_score, void* ws, size_t ws_bytes,
                                              void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_e4m3_dims(dims));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  const E4m3Plan plan = e4m3_plan(n, dims->D);
  if (plan.score.vtiles > 65535) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(hidden, n.N));
  JET_TRY(check_ptr(w4, n.V));
  if ((reinterpret_cast<uintptr_t>(w4) & 31u) != 0) return JET_ERR_ALIGN;  // the TMA's 4-bit map
  JET_TRY(check_ptr(w_scale, n.V));
  JET_TRY(check_ptr(tok_logprob, n.T));
  JET_TRY(check_ptr(cand_score, n.C));
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  int* status = jet::device_status_ptr();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* h_q = static_cast<uint8_t*>(ws) + plan.hq_off;
  float* h_scale = reinterpret_cast<float*>(static_cast<char*>(ws) + plan.hs_off);
  JET_TRY(cuda_status(jet::launch_quantize_e4m3(hidden, n.N, dims->D, h_q, h_scale, st)));
  JET_TRY(cuda_status(jet::launch_lmhead_w4(*lay, *dims, plan.score, h_q, h_scale, w4, w_scale,
                                            ws, status, st)));
  return cuda_status(
      jet::launch_score_finish(*lay, plan.score, ws, tok_logprob, cand_score, status, st));
}

extern "C" size_t jet_mxfp8_bytes(int64_t V, int64_t D) {
  if (V < 1 || D < 16 || D % 16 != 0 || V > (int64_t(1) << 30) || D > (int64_t(1) << 20)) return 0;
  return mx_weight_bytes(V, D);
}

extern "C" jet_status jet_quantize_mxfp8(const void* w, int64_t V, int64_t D, uint8_t* out,
                                         void* stream) {
  if (V < 1) return JET_ERR_ARG;
  if (D < 16 || D % 16 != 0) return JET_ERR_SHAPE;
  if (V > (int64_t(1) << 30) || D > (int64_t(1) << 20)) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(w, V));
  JET_TRY(check_ptr(out, V));
  const int vtiles = int((V + 127) / 128);
  uint8_t* sf = out + ((size_t(V) * size_t(D) + 255) & ~size_t(255));
  return cuda_status(jet::launch_quantize_mx(w, int(V), int(D), vtiles * 128, 128, 1, out, sf,
                                             static_cast<cudaStream_t>(stream)));
}

extern "C" size_t jet_workspace_bytes_mxfp8(const jet_sizes* n, const jet_dims* d) {
  if (!n || !d || n->R < 0 || n->N < 0 || n->V < 1 || d->D < 16) return 0;
  size_t a = 0;
  if (d->Hq > 0 && d->Hkv > 0 && d->Hq % d->Hkv == 0 && d->d > 0) a = jet::attn_plan(*n, *d).bytes;
  const size_t b = mx_plan(*n, d->D).bytes;
  return a > b ? a : b;
}

extern "C" jet_status jet_score_candidates_mxfp8(const jet_layout* lay, const jet_dims* dims,
                                                 const void* hidden, const uint8_t* w_mx,
                                                 float* tok_logprob, float* cand_score, void* ws,
                                                 size_t ws_bytes, void* stream) {
  JET_TRY(check_layout(lay));
  JET_TRY(check_e4m3_dims(dims));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  const MxPlan plan = mx_plan(n, dims->D);
  if (plan.score.vtiles > 65535) return JET_ERR_CAPACITY;
  JET_TRY(check_ptr(hidden, n.N));
  JET_TRY(check_ptr(w_mx, n.V));
  JET_TRY(check_ptr(tok_logprob, n.T));
  JET_TRY(check_ptr(cand_score, n.C));
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  int* status = jet::device_status_ptr();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* h_q = static_cast<uint8_t*>(ws) + plan.hq_off;
  uint8_t* h_sf = static_cast<uint8_t*>(ws) + plan.hsf_off;
  // the hidden states into codes and per-token-tile scale-factor chunks
  JET_TRY(cuda_status(jet::launch_quantize_mx(hidden, n.N, dims->D, plan.n_tt * 256, plan.Nt, 2,
                                              h_q, h_sf, st)));
  const uint8_t* w_sf = w_mx + ((size_t(n.V) * size_t(dims->D) + 255) & ~size_t(255));
  JET_TRY(cuda_status(jet::launch_lmhead_mx(*lay, *dims, plan.score, h_q, h_sf, w_mx, w_sf, ws,
                                            status, st)));
  return cuda_status(
      jet::launch_score_finish(*lay, plan.score, ws, tok_logprob, cand_score, status, st));
}

namespace {

// scratch of jet_stack_forward (offsets 256-byte aligned)
struct StackPlan {
  size_t h, z, q, kc, vc, lqa, lqf, lk, lv, al, be, o, u, attn, part, bytes;
  jet::AttnPlan attn_plan;
  bool full_ok, lin_ok;
};

StackPlan stack_plan(const jet_sizes& n, const jet_dims& d, int Dff) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  StackPlan p{};
  const size_t N = size_t(n.N), F = size_t(n.N - n.R), b = 2;
  p.full_ok = check_attn_dims(&d) == JET_OK;
  p.lin_ok = check_fork_dims(&d) == JET_OK && d.Hl % 2 == 0;
  const size_t zf = p.full_ok ? size_t(d.Hq + 2 * d.Hkv) * d.d : 0;
  const size_t zl = p.lin_ok ? size_t(d.Hl) * (2 * d.dk + d.dv) + 2 * d.Hl : 0;
  const size_t ow = std::max(p.full_ok ? size_t(d.Hq) * d.d : 0,
                             p.lin_ok ? size_t(d.Hl) * d.dv : 0);
  size_t at = 0;
  auto take = [&](size_t bytes) {
    const size_t off = at;
    at += up(bytes);
    return off;
  };
  p.h = take(N * d.D * b);
  p.z = take(N * std::max(zf, zl) * b);
  p.o = take(N * ow * b);
  p.u = take(N * size_t(Dff) * b);
  // split-K partials of the largest projection that splits
  size_t part = jet::proj_partial_bytes(n.N, 2 * Dff, d.D);
  part = std::max(part, jet::proj_partial_bytes(n.N, d.D, Dff));
  if (zf) {
    part = std::max(part, jet::proj_partial_bytes(n.N, int(zf), d.D));
    part = std::max(part, jet::proj_partial_bytes(n.N, d.D, d.Hq * d.d));
  }
  if (zl) {
    part = std::max(part, jet::proj_partial_bytes(n.N, int(zl), d.D));
    part = std::max(part, jet::proj_partial_bytes(n.N, d.D, d.Hl * d.dv));
  }
  p.part = take(part);
  if (p.full_ok) {
    p.q = take(N * d.Hq * d.d * b);
    p.kc = take(F * d.Hkv * d.d * b);
    p.vc = take(F * d.Hkv * d.d * b);
    p.attn_plan = jet::attn_plan(n, d);
    p.attn = take(p.attn_plan.bytes);
  }
  if (p.lin_ok) {
    p.lqa = take(N * d.Hl * d.dk * b);
    p.lqf = take(F * d.Hl * d.dk * b);
    p.lk = take(F * d.Hl * d.dk * b);
    p.lv = take(F * d.Hl * d.dv * b);
    p.al = take(F * d.Hl * 4);
    p.be = take(F * d.Hl * 4);
  }
  p.bytes = at;
  return p;
}

}  // namespace

extern "C" size_t jet_stack_workspace_bytes(const jet_sizes* n, const jet_dims* d, int32_t Dff) {
  if (!n || !d || n->R < 0 || n->N < n->R || d->D < 16 || Dff < 64 || Dff % 64 != 0) return 0;
  return stack_plan(*n, *d, Dff).bytes;
}

extern "C" jet_status jet_stack_forward(const jet_layout* lay, const jet_dims* dims,
                                        const jet_stack* stack, const void* x0, void* x,
                                        void* ws, size_t ws_bytes, void* stream) {
  JET_TRY(check_layout(lay));
  if (!dims || !stack) return JET_ERR_ARG;
  JET_TRY(check_dtype(dims));
  if (dims->dtype != JET_DTYPE_BF16) return JET_ERR_UNSUPPORTED;
  if (dims->D < 16 || dims->D % 16 != 0) return JET_ERR_SHAPE;
  if (stack->L < 0 || (stack->L > 0 && !stack->layers)) return JET_ERR_ARG;
  if (stack->Dff < 64 || stack->Dff % 64 != 0) return JET_ERR_SHAPE;
  if (stack->rule != JET_RECUR_DELTA && stack->rule != JET_RECUR_GLA) return JET_ERR_ARG;
  const jet_sizes& n = lay->n;
  const long long N = n.N;
  const StackPlan plan = stack_plan(n, *dims, stack->Dff);
  // validate every layer before the first launch
  for (int l = 0; l < stack->L; ++l) {
    const jet_stack_layer& Ly = stack->layers[l];
    if (Ly.kind == JET_LAYER_FULL) {
      JET_TRY(check_attn_dims(dims));
      if ((long long)n.R * dims->Hkv > 65535) return JET_ERR_CAPACITY;
      JET_TRY(check_ptr(Ly.k_pre, n.total_prefix));
      JET_TRY(check_ptr(Ly.v_pre, n.total_prefix));
    } else if (Ly.kind == JET_LAYER_LINEAR) {
      JET_TRY(check_fork_dims(dims));
      if (dims->Hl % 2 != 0) return JET_ERR_UNSUPPORTED;
      if (n.R > 65535 || dims->Hl > 65535 || dims->dv > 1024) return JET_ERR_CAPACITY;
      JET_TRY(check_ptr(Ly.s_prefix, n.R));
    } else {
      return JET_ERR_ARG;
    }
    JET_TRY(check_ptr(Ly.g1, 1));
    JET_TRY(check_ptr(Ly.g2, 1));
    JET_TRY(check_ptr(Ly.w_mix, 1));
    JET_TRY(check_ptr(Ly.w_o, 1));
    JET_TRY(check_ptr(Ly.w_gu, 1));
    JET_TRY(check_ptr(Ly.w_d, 1));
  }
  if (n.R == 0) return JET_OK;
  JET_TRY(check_ptr(x0, N));
  JET_TRY(check_ptr(x, N));
  if (!ws || ws_bytes < plan.bytes) return JET_ERR_WORKSPACE;
  if (!aligned16(ws)) return JET_ERR_ALIGN;
  if (N > 65535 * 8 || (long long)N * dims->D > INT32_MAX) return JET_ERR_CAPACITY;
  int* status = jet::device_status_ptr();
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* w = static_cast<char*>(ws);
  float* part = reinterpret_cast<float*>(w + plan.part);
  const int D = dims->D, Dff = stack->Dff;
  const size_t xbytes = size_t(N) * D * 2;
  if (x != x0)
    JET_TRY(cuda_status(cudaMemcpyAsync(x, x0, xbytes, cudaMemcpyDeviceToDevice, st)));
  for (int l = 0; l < stack->L; ++l) {
    const jet_stack_layer& Ly = stack->layers[l];
    const bool full = Ly.kind == JET_LAYER_FULL;
    // h = RMSNorm(x; g1): the previous layer's down projection already wrote it
    if (l == 0)
      JET_TRY(cuda_status(jet::launch_rmsnorm(x, Ly.g1, int(N), D, 1e-6f, w + plan.h, st)));
    const int zw = full ? (dims->Hq + 2 * dims->Hkv) * dims->d
                        : dims->Hl * (2 * dims->dk + dims->dv) + 2 * dims->Hl;
    int ow;
    if (full) {
      // the q/k/v projection and its split into the step's query and candidate
      // key/value buffers in one pass over its partials
      const int qw = dims->Hq * dims->d, kw = dims->Hkv * dims->d;
      JET_TRY(cuda_status(jet::launch_proj_qkv(*lay, w + plan.h, D, Ly.w_mix, qw, kw, w + plan.z,
                                               w + plan.q, w + plan.kc, w + plan.vc, part, status,
                                               st)));
      JET_TRY(cuda_status(jet::launch_prefix_attend(*lay, *dims, plan.attn_plan, w + plan.q,
                                                    Ly.k_pre, Ly.v_pre, w + plan.kc,
                                                    w + plan.vc, w + plan.o, w + plan.attn,
                                                    status, st)));
      ow = qw;
    } else {
      float* al = reinterpret_cast<float*>(w + plan.al);
      float* be = reinterpret_cast<float*>(w + plan.be);
      // the mixer projection and the gates (q, normalised k, v, decay and write
      // strength) in one pass over its partials
      JET_TRY(cuda_status(jet::launch_proj_gates(*lay, w + plan.h, D, Ly.w_mix, zw, w + plan.z,
                                                 dims->Hl, dims->dv, w + plan.lqa, w + plan.lqf,
                                                 w + plan.lk, w + plan.lv, al, be, part, status,
                                                 st)));
      // fed rows through the fork, shared rows from the prefix states: all N
      // rows of the mixer output
      JET_TRY(cuda_status(jet::launch_fork_state(*lay, *dims, stack->rule, Ly.s_prefix,
                                                 w + plan.lqf, w + plan.lk, w + plan.lv, al, be,
                                                 w + plan.o, nullptr, status, st,
                                                 w + plan.lqa)));
      ow = dims->Hl * dims->dv;
    }
    // x += W_o o, then h = RMSNorm(x; g2)
    JET_TRY(cuda_status(jet::launch_proj(jet::kProjResid, w + plan.o, int(N), ow, ow, Ly.w_o, D,
                                         x, D, x, part, status, st, Ly.g2, 1e-6f, w + plan.h)));
    JET_TRY(cuda_status(jet::launch_proj(jet::kProjSwiGLU, w + plan.h, int(N), D, D, Ly.w_gu,
                                         2 * Dff, w + plan.u, Dff, nullptr, part, status,
                                         st)));
    // x += W_d u, then the next layer's h = RMSNorm(x; g1')
    const bool next = l + 1 < stack->L;
    JET_TRY(cuda_status(jet::launch_proj(jet::kProjResid, w + plan.u, int(N), Dff, Dff, Ly.w_d,
                                         D, x, D, x, part, status, st,
                                         next ? stack->layers[l + 1].g1 : nullptr, 1e-6f,
                                         next ? w + plan.h : nullptr)));
  }
  return JET_OK;
}

extern "C" jet_status jet_decide(const jet_layout* lay, int32_t mode, const float* cand_score,
                                 float* q, int32_t* choice, float* value, void* stream) {
  JET_TRY(check_layout(lay));
  if (mode != JET_DECIDE_ARGMAX && mode != JET_DECIDE_BINARY && mode != JET_DECIDE_ORDINAL)
    return JET_ERR_ARG;
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  if (mode == JET_DECIDE_BINARY && (n.min_cand != 2 || n.max_cand != 2)) return JET_ERR_SHAPE;
  JET_TRY(check_ptr(cand_score, n.C));
  JET_TRY(check_ptr(q, n.C));
  JET_TRY(check_ptr(choice, n.R));
  JET_TRY(check_ptr(value, n.R));
  return cuda_status(jet::launch_decide(*lay, mode, cand_score, q, choice, value,
                                        jet::device_status_ptr(),
                                        static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_evaluate(const jet_layout* lay, const float* cand_score,
                                   const int32_t* choice, const uint8_t* gold, float* nll,
                                   int32_t* correct, void* stream) {
  JET_TRY(check_layout(lay));
  const jet_sizes& n = lay->n;
  if (n.R == 0) return JET_OK;
  JET_TRY(check_ptr(cand_score, n.C));
  JET_TRY(check_ptr(choice, n.R));
  JET_TRY(check_ptr(gold, n.C));
  JET_TRY(check_ptr(nll, n.R));
  JET_TRY(check_ptr(correct, n.R));
  return cuda_status(jet::launch_evaluate(*lay, cand_score, choice, gold, nll, correct,
                                          jet::device_status_ptr(),
                                          static_cast<cudaStream_t>(stream)));
}

extern "C" jet_status jet_device_status(void* stream, jet_status* out) {
  if (!out) return JET_ERR_ARG;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return JET_ERR_CUDA;
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, jet::g_status_word, sizeof(int)) != cudaSuccess) return JET_ERR_CUDA;
  const int zero = 0;
  if (cudaMemcpyToSymbol(jet::g_status_word, &zero, sizeof(int)) != cudaSuccess) return JET_ERR_CUDA;
  *out = v;
  return JET_OK;
}

extern "C" uint64_t jet_set_wait_budget_ns(uint64_t ns) {
  return jet::g_wait_ns.exchange(ns ? ns : jet::kDefaultWaitNs);
}

extern "C" uint64_t jet_launch_count(void) { return jet::g_launches.load(); }

extern "C" int32_t jet_set_test_stall(int32_t on) { return jet::g_test_stall.exchange(on ? 1 : 0); }
