// Internal declarations shared by the CUDA translation units of libjet.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "jet.h"

namespace jet {

// ---- per-device status word -------------------------------------------------
// Device address of the current device's status word (set up once per device);
// nullptr when the address cannot be obtained.
int* device_status_ptr();

// ---- workspace plans -----------------------------------------------------------
constexpr int kVocabTile = 128;  // vocabulary entries per LM-head partial
// 4-bit weights, per (128 vocabulary rows, 128-element K slice): 128 x 64
// bytes of packed E2M1 codes (in the row-major code region) and a 512-byte
// chunk of UE8M0 block scale factors (in the scale region after it)
constexpr int kW4CodeBytes = kVocabTile * 64;
constexpr int kW4ScaleBytes = 512;
constexpr int kW4TileBytes = kW4CodeBytes + kW4ScaleBytes;

struct AttnPlan {
  int splits;    // prefix chunks per (request, key/value head)
  int chunk;     // prefix keys per chunk (multiple of 32)
  int qgroups;   // query-vector groups per (request, key/value head)
  size_t bytes;  // workspace bytes
};
AttnPlan attn_plan(const jet_sizes& n, const jet_dims& d);

struct ScorePlan {
  int vtiles;          // ceil(V / kVocabTile)
  size_t part_off;     // float2 partials [N][vtiles]
  size_t ztgt_off;     // float z_tgt[T]
  size_t lse_off;      // float lse[N]
  size_t bytes;
};
ScorePlan score_plan(const jet_sizes& n);

// ---- host-side run settings -------------------------------------------------------
// Budget in nanoseconds of one bounded wait inside the tensor-core kernels
// (jet_set_wait_budget_ns; 2 s unless set), read at every launch and passed
// to the kernel as an argument.
uint64_t wait_budget_ns();
// Test hook (jet_set_test_stall): nonzero makes the tensor-core kernels
// launched afterwards withhold their first load, so that a wait nothing will
// satisfy runs out its budget.
int test_stall();
// Counts one kernel launch of this library (jet_launch_count).
void note_launch();

// ---- launches ------------------------------------------------------------------
// Stream-ordered launch with programmatic stream serialization: the kernel may
// begin (up to its pdl_begin()) while the previous kernel of the stream ends,
// which hides the launch latency between the dependent kernels of a step.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr{};
  attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr.val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
  if (e == cudaSuccess) note_launch();
  return e;
}

// The same as a grid of clusters of two CTAs (grid.x even).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_pairs(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2]{};
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, args...);
  if (e == cudaSuccess) note_launch();
  return e;
}

// ---- kernel launchers (stream-ordered; return the launch error) ---------------
cudaError_t launch_prefix_attend(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                                 const void* q, const void* k_pre, const void* v_pre,
                                 const void* k_cand, const void* v_cand, void* o, void* ws,
                                 int* status, cudaStream_t st);

// bf16 cascade attention on the tensor cores (attend_tc.cu): prefix chunks and
// the candidates' own keys, plus the chunk combine; query vectors per CTA
int attn_tc_block();
cudaError_t launch_attend_tc(const jet_layout& lay, const jet_dims& d, const AttnPlan& plan,
                             const void* q, const void* k_pre, const void* v_pre,
                             const void* k_cand, const void* v_cand, void* o, float* o_part,
                             float2* ml_part, int* status, cudaStream_t st);

// the prefix scan of the recurrent state (prefill of a linear-attention layer)
cudaError_t launch_prefill_state(const jet_layout& lay, const jet_dims& d, int rule,
                                 const float* s_init, const void* q, const void* k, const void* v,
                                 const float* alpha, const float* beta, void* o, float* s_out,
                                 int* status, cudaStream_t st);
// rule: JET_RECUR_DELTA or JET_RECUR_GLA
// the chunked scan on the tensor cores (scan_tc.cu): bf16 inputs, dk = dv = 128
bool scan_tc_supported(const jet_dims& d);
cudaError_t launch_scan_tc(const jet_layout& lay, const jet_dims& d, int rule,
                           const float* s_init, const void* q, const void* k, const void* v,
                           const float* alpha, const float* beta, void* o, float* s_out,
                           int* status, cudaStream_t st);
// causal self-attention over every request's prefix (bf16, tensor cores);
// the workspace holds the work list
size_t prefill_workspace_bytes(const jet_sizes& n, const jet_dims& d);
cudaError_t launch_prefill_tc(const jet_layout& lay, const jet_dims& d, const void* q,
                              const void* k, const void* v, void* o, void* ws, int* status,
                              cudaStream_t st);

// q_rows (optional, every row's q [N, Hl, dk]): o then covers all N rows, the
// shared rows reading the prefix states (o = S_r^T q / sqrt(dk)) and fed token
// f at row f + r + 1; without it o holds the fed tokens only
cudaError_t launch_fork_state(const jet_layout& lay, const jet_dims& d, int rule,
                              const float* s_prefix, const void* q, const void* k, const void* v,
                              const float* alpha, const float* beta, void* o, float* s_fork,
                              int* status, cudaStream_t st, const void* q_rows = nullptr);

// logits partials: writes part[N][vtiles] (m, s) in base 2 - m = max_v z log2(e),
// s = sum_v 2^(z log2(e) - m) over the tile - and z_tgt[T]
cudaError_t launch_lmhead_simt(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                               const void* hidden, const void* w_lm, void* ws, int* status,
                               cudaStream_t st);
cudaError_t launch_lmhead_tc(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const void* hidden, const void* w_lm, void* ws, int* status,
                             cudaStream_t st);
// e4m3 codes [N, D] / [V, D] with float32 scales per token / vocabulary row
cudaError_t launch_lmhead_e4m3(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                               const uint8_t* h_q, const float* h_scale, const uint8_t* w_q,
                               const float* w_scale, void* ws, int* status, cudaStream_t st);
// ---- decoder stacks -------------------------------------------------------------
enum { kProjStore = 0, kProjResid = 1, kProjSwiGLU = 2 };
// out[N, O] = epilogue(x[N, K] w[O, K]^T) on the tensor cores (bf16, f32 accumulate);
// ldx / ldo are the row strides of x and out in elements; res (kProjResid) may be
// out; part: f32 scratch of proj_partial_bytes(N, O, K) bytes for a split K (null:
// no split); kProjResid with norm_h: also h = RMSNorm(out; norm_g, norm_eps),
// the next layer input, in the same pass where the K split allows
cudaError_t launch_proj(int epi, const void* x, int N, int K, int ldx, const void* w, int O,
                        void* out, int ldo, const void* res, float* part, int* status,
                        cudaStream_t st, const void* norm_g = nullptr, float norm_eps = 0.f,
                        void* norm_h = nullptr);
size_t proj_partial_bytes(int N, int O, int K);
// a linear layer's mixer projection z = x w^T (O = Hl (2 dk + dv) + 2 Hl) and
// its gates (launch_gates) in one go: with a K split the partials are reduced
// straight into the gates' outputs, without z
cudaError_t launch_proj_gates(const jet_layout& lay, const void* x, int K, const void* w, int O,
                              void* z, int Hl, int dv, void* lq_all, void* lq, void* lk, void* lv,
                              float* alpha, float* beta, float* part, int* status,
                              cudaStream_t st);
// a full-attention layer's q/k/v projection (O = qw + 2 kw) and its split into q
// and the fed rows' k and v (launch_split_qkv) in one go, likewise
cudaError_t launch_proj_qkv(const jet_layout& lay, const void* x, int K, const void* w, int qw,
                            int kw, void* z, void* q, void* kc, void* vc, float* part,
                            int* status, cudaStream_t st);
cudaError_t launch_reduce_qkv(const jet_layout& lay, const float* part, int splits, int qw,
                              int kw, void* q, void* kc, void* vc, int* status, cudaStream_t st);
cudaError_t launch_reduce_gates(const jet_layout& lay, const float* part, int splits, int Hl,
                                int dv, void* lq_all, void* lq, void* lk, void* lv,
                                float* alpha, float* beta, int* status, cudaStream_t st);
cudaError_t launch_rmsnorm(const void* x, const void* g, int N, int D, float eps, void* h,
                           cudaStream_t st);
cudaError_t launch_split_qkv(const jet_layout& lay, const void* z, int qw, int kw, void* q,
                             void* kc, void* vc, int* status, cudaStream_t st);
cudaError_t launch_gates(const jet_layout& lay, const void* z, int Hl, int dv, void* lq_all,
                         void* lq, void* lk, void* lv, float* alpha, float* beta, int* status,
                         cudaStream_t st);

// the LM head on tiled 4-bit weights (w4) and e4m3 hidden codes
cudaError_t launch_lmhead_w4(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const uint8_t* h_q, const float* h_scale, const uint8_t* w4,
                             const float* w_scale, void* ws, int* status, cudaStream_t st);
// 4-bit quantisation of a bf16 matrix [V, D] into the tiled layout, scales [V]
cudaError_t launch_quantize_w4(const void* x, int V, int D, uint8_t* w4, float* scale,
                               cudaStream_t st);
// MXFP8 quantisation (e4m3 codes, a UE8M0 factor per 32-element block) of
// the bf16 matrix x [rows, D]: `slots` row slots in groups of 128 * halves,
// slot rs of group g being row g * tile_rows + rs (rs < tile_rows); codes
// row-major [rows, D], factors in 512-byte chunks per (group, K slice, half)
cudaError_t launch_quantize_mx(const void* x, int rows, int D, int slots, int tile_rows,
                               int halves, uint8_t* codes, uint8_t* sf, cudaStream_t st);
// the MXFP8 LM head's token tiles: at most 224 rows (a multiple of 16) each
void mx_token_tiling(int N, int* Nt, int* n_tt);
// the LM head on MXFP8 weights (codes [V, D], factors per 128-row tile and K
// slice) and MXFP8 hidden states (codes [N, D], factors per token tile and K
// slice, two chunks each)
cudaError_t launch_lmhead_mx(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                             const uint8_t* h_q, const uint8_t* h_sf, const uint8_t* w_q,
                             const uint8_t* w_sf, void* ws, int* status, cudaStream_t st);
// per-row e4m3 quantisation of a bf16 matrix [rows, D] (D multiple of 16)
cudaError_t launch_quantize_e4m3(const void* x, int rows, int D, uint8_t* q, float* scale,
                                 cudaStream_t st);
cudaError_t launch_lmhead(const jet_layout& lay, const jet_dims& d, const ScorePlan& plan,
                          const void* hidden, const void* w_lm, void* ws, int* status,
                          cudaStream_t st);

// lse per row, then l_{c,t} and s(c|x)
cudaError_t launch_score_finish(const jet_layout& lay, const ScorePlan& plan, void* ws,
                                float* tok_logprob, float* cand_score, int* status,
                                cudaStream_t st);

cudaError_t launch_evaluate(const jet_layout& lay, const float* cand_score, const int32_t* choice,
                            const uint8_t* gold, float* nll, int32_t* correct, int* status,
                            cudaStream_t st);

cudaError_t launch_decide(const jet_layout& lay, int mode, const float* cand_score, float* q,
                          int32_t* choice, float* value, int* status, cudaStream_t st);

}  // namespace jet
