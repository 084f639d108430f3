/*
 * jet.h - C ABI of the JET teacher-forced candidate-scoring step on GB300
 * (sm_103a).
 *
 * JET (Justification Evaluation in Transformer) picks an answer from a
 * finite candidate set by the candidates' teacher-forced likelihoods under a
 * language model (Sec. 3). For a question context x, candidates
 * y_c = (y_{c,1} .. y_{c,m_c}) and vocabulary V, one step computes
 *
 *   attention   shared-prefix cascade attention: every candidate row attends
 *               to the request's prefix K/V plus its own earlier candidate
 *               tokens (Sec. 4.1)                        -> jet_prefix_attend
 *   fork        per-candidate continuation of an unmodified copy of the
 *               prefix recurrent state (Sec. 4.1)        -> jet_fork_state
 *   score       l_{c,t} = log p(y_{c,t} | x, y_{c,<t}) over the full
 *               vocabulary (Eq. 1, Eq. 2) and s(c|x) = sum_t l_{c,t} (Eq. 3);
 *               logits never leave the chip (Sec. 4.2)   -> jet_score_candidates
 *   decide      q(c) = softmax over candidates (Eq. 4), argmax choice (Eq. 5),
 *               binary q(true) or ordinal expectation (Sec. 3.3) -> jet_decide
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every function returns a jet_status; 0 (JET_OK) means success. Nothing is
 *   launched when a call returns an error. The library never allocates
 *   memory, never synchronises a stream (except jet_device_status), never
 *   prints and never exits the process.
 * - Tensor arguments are DEVICE pointers owned by the caller, 16-byte
 *   aligned, row-major and dense, in the element type jet_dims.dtype names
 *   (float32 or bf16) unless stated otherwise.
 * - A layout's int32 arrays live where the call needs them: host memory for
 *   jet_layout_build, device memory for the compute calls (copy the words
 *   buffer once and bind it with jet_layout_bind).
 * - Work is enqueued on `stream` (a cudaStream_t passed as void*; NULL means
 *   the legacy default stream) and runs asynchronously.
 * - Kernels check every index they read from a device layout and skip an
 *   out-of-range access instead of faulting; they then record
 *   JET_ERR_DEVICE in a per-device status word that jet_device_status reads.
 *
 * Row layout (Sec. 3.1, Eq. 1; Sec. 4.1)
 * --------------------------------------
 * Request r owns n_r = 1 + sum_c (m_c - 1) consecutive query rows. Its first
 * ("shared") row is the last prefix position: its logits condition on x alone
 * and give p(y_{c,1} | x) for every candidate c. Then, candidate by candidate,
 * one row per fed token y_{c,t}, t = 1 .. m_c - 1; the row fed with y_{c,t}
 * predicts y_{c,t+1}. y_{c,m_c} is a target only. N = sum_r n_r rows,
 * T = sum_c m_c targets, C = sum_r C_r candidates, F = N - R fed tokens.
 * Candidate tensors indexed by fed token use row order with the shared rows
 * left out: the fed token of row n of request r has index n - r - 1.
 */
#ifndef JET_H
#define JET_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define JET_ABI_VERSION 1

typedef int32_t jet_status;
enum {
  JET_OK = 0,
  JET_ERR_ARG = 1,         /* null pointer or invalid scalar argument          */
  JET_ERR_SHAPE = 2,       /* inconsistent sizes (Hq % Hkv != 0, m_c < 1, ...)  */
  JET_ERR_RANGE = 3,       /* a token id outside [0, V)                          */
  JET_ERR_ALIGN = 4,       /* a device pointer that is not 16-byte aligned       */
  JET_ERR_WORKSPACE = 5,   /* workspace null or smaller than jet_workspace_bytes */
  JET_ERR_CAPACITY = 6,    /* a size beyond what the kernels index (2^31 elems)  */
  JET_ERR_UNSUPPORTED = 7, /* dtype or head dimension the kernels do not handle */
  JET_ERR_CUDA = 8,        /* a CUDA runtime call or launch failed               */
  JET_ERR_TIMEOUT = 9,     /* a bounded device-side wait gave up                 */
  JET_ERR_DEVICE = 10      /* a kernel met an out-of-range index in a layout     */
};

enum { JET_DTYPE_F32 = 0, JET_DTYPE_BF16 = 1 };

/* recurrences of the linear-attention fork (the paper names none; see
 * jet_fork_state_rule) */
enum { JET_RECUR_DELTA = 0, JET_RECUR_GLA = 1 };

/* decision rules of Sec. 3.3 / Eq. 5 */
enum { JET_DECIDE_ARGMAX = 0, JET_DECIDE_BINARY = 1, JET_DECIDE_ORDINAL = 2 };

/* Sizes of one batch; filled by jet_layout_plan. */
typedef struct jet_sizes {
  int32_t R;            /* requests (contexts x)                          */
  int32_t C;            /* candidates, sum_r C_r                          */
  int32_t N;            /* query rows, sum_r n_r                          */
  int32_t T;            /* targets, sum_c m_c                             */
  int32_t V;            /* vocabulary size |V|                            */
  int32_t total_prefix; /* sum_r P_r                                      */
  int32_t max_prefix;   /* max_r P_r                                      */
  int32_t min_cand;     /* min_r C_r                                      */
  int32_t max_cand;     /* max_r C_r                                      */
  int32_t max_rows;     /* max_r n_r                                      */
  int32_t max_len;      /* max_c m_c                                      */
  int32_t reserved;
} jet_sizes;

/*
 * The integer layout of a batch (Sec. 3.1, Eq. 1; Sec. 4.1). All arrays are
 * int32 and point into one "words" buffer of jet_layout_words() entries.
 *   prefix_offset[R+1]   request r's prefix keys are [prefix_offset[r], prefix_offset[r+1])
 *                        of the packed prefix K/V
 *   cand_offset[R+1]     request r's candidates are [cand_offset[r], cand_offset[r+1])
 *   row_offset[R+1]      request r's rows; row_offset[r] is its shared row
 *   cand_row_offset[C+1] first fed row of candidate c (its m_c - 1 fed rows
 *                        are consecutive); entry C is N
 *   tgt_offset[C+1]      candidate c's targets y_{c,1..m_c} are
 *                        [tgt_offset[c], tgt_offset[c+1])
 *   target_ids[T]        y_{c,t} in candidate order
 *   tgt_row[T]           the row whose logits predict target j
 *   row_req[N]           request of row n
 *   row_cand[N]          candidate of row n, -1 for a shared row
 *   row_pos[N]           t of the token fed at row n, 0 for a shared row
 *   row_tgt_offset[N+1], row_tgt_index[T]
 *                        the targets predicted by row n, in increasing index
 *   req_order[R]         the requests by decreasing prefix length (ties: lower
 *                        index first); the attention kernels hand out long
 *                        prefixes first
 */
typedef struct jet_layout {
  jet_sizes n;
  const int32_t* prefix_offset;
  const int32_t* cand_offset;
  const int32_t* row_offset;
  const int32_t* cand_row_offset;
  const int32_t* tgt_offset;
  const int32_t* target_ids;
  const int32_t* tgt_row;
  const int32_t* row_req;
  const int32_t* row_cand;
  const int32_t* row_pos;
  const int32_t* row_tgt_offset;
  const int32_t* row_tgt_index;
  const int32_t* req_order;
} jet_layout;

/* Model dimensions of the step (and one launch limit). */
typedef struct jet_dims {
  int32_t dtype; /* JET_DTYPE_*: element type of q, k, v, o, hidden, w_lm    */
  int32_t Hq;    /* attention query heads                                    */
  int32_t Hkv;   /* attention key/value heads; query head h uses
                    key/value head h / (Hq / Hkv) (grouped-query attention) */
  int32_t d;     /* attention head dimension: 64, 128 or 256                  */
  int32_t D;     /* LM-head hidden size (multiple of 8)                       */
  int32_t Hl;    /* linear-attention heads (0 when the model has none)        */
  int32_t dk;    /* linear-attention key dimension: 128                       */
  int32_t dv;    /* linear-attention value dimension: multiple of 32, <= 256 */
  int32_t max_sms; /* at most this many SMs for the persistent LM-head kernel
                      (0: all of them). An HBM-bound LM head reaches the
                      bandwidth roof with fewer SMs; leaving some free lets a
                      caller run other work (the next batch's attention) on
                      another stream at the same time. */
} jet_dims;

/* ABI version of the loaded library (JET_ABI_VERSION it was built with). */
int32_t jet_abi_version(void);

/* Static description of a status code; never NULL. */
const char* jet_status_string(jet_status s);

/*
 * jet_layout_plan - sizes of a batch, from its structure (host only).
 * prefix_len[R] = P_r >= 1, n_cand[R] = C_r >= 1, cand_len[C] = m_c >= 1 in
 * request order, V >= 1. Errors: JET_ERR_ARG (null, R < 0, V < 1),
 * JET_ERR_SHAPE (a count below 1), JET_ERR_CAPACITY (a total beyond int32).
 */
jet_status jet_layout_plan(int32_t R, const int32_t* prefix_len, const int32_t* n_cand,
                           const int32_t* cand_len, int32_t V, jet_sizes* out);

/* Number of int32 words a layout of these sizes occupies. */
size_t jet_layout_words(const jet_sizes* n);

/*
 * jet_layout_build - the teacher-forced layout (host only, Sec. 3.1, Eq. 1;
 * Sec. 4.1). target_ids[T] lists y_{c,1..m_c} for every candidate in request
 * order; each must lie in [0, V) (else JET_ERR_RANGE). `words` is a caller
 * buffer of n_words >= jet_layout_words() int32 (else JET_ERR_WORKSPACE);
 * `out` is bound to it. The words may then be copied verbatim to the device
 * and bound with jet_layout_bind.
 */
jet_status jet_layout_build(int32_t R, const int32_t* prefix_len, const int32_t* n_cand,
                            const int32_t* cand_len, const int32_t* target_ids, int32_t V,
                            int32_t* words, size_t n_words, jet_layout* out);

/* jet_layout_bind - point a layout's arrays into a (host or device) copy of
 * the words buffer. Does not read the words. */
jet_status jet_layout_bind(const jet_sizes* n, const int32_t* words, jet_layout* out);

/* Workspace bytes jet_prefix_attend and jet_score_candidates need for a batch
 * of these sizes (the larger of the two; one buffer serves both calls when
 * they run one after the other on a stream). 0 on invalid arguments. */
size_t jet_workspace_bytes(const jet_sizes* n, const jet_dims* dims);

/*
 * jet_prefix_attend - shared-prefix cascade attention (Sec. 4.1, Fig. 1
 * "KV-cache text models"; scale 1/sqrt(d), no positional encoding).
 *   q       [N, Hq, d]           query of every row
 *   k_pre   [total_prefix, Hkv, d], v_pre likewise: packed prefix K/V
 *   k_cand  [F, Hkv, d], v_cand likewise: K/V of the fed candidate tokens
 *   o       [N, Hq, d]           output
 * The shared row of request r attends to its P_r prefix keys; the row fed
 * with y_{c,t} attends to the prefix and to y_{c,1..t} of its own candidate.
 * The prefix K/V of a request is read once per key/value head by all of the
 * request's rows. Accumulation is float32; o is written in dims.dtype.
 * ws/ws_bytes: scratch of at least jet_workspace_bytes().
 */
jet_status jet_prefix_attend(const jet_layout* lay, const jet_dims* dims, const void* q,
                             const void* k_pre, const void* v_pre, const void* k_cand,
                             const void* v_cand, void* o, void* ws, size_t ws_bytes,
                             void* stream);

/*
 * jet_prefill_attend - the prefill before the scoring step: causal
 * self-attention over every request's prefix (Sec. 4.1: the shared prefix is
 * evaluated once and its K/V reused by every candidate; scale 1/sqrt(d), no
 * positional encoding, grouped-query heads as in jet_prefix_attend).
 *   q     [total_prefix, Hq, d]    queries of the prefix positions
 *   k, v  [total_prefix, Hkv, d]   the prefix K/V (what jet_prefix_attend reads)
 *   o     [total_prefix, Hq, d]    position p of request r attends to r's keys 0..p
 * bf16 only (else JET_ERR_UNSUPPORTED), d in {64, 128, 256}. Uses the layout's
 * prefix sizes only. ws/ws_bytes: scratch of at least
 * jet_prefill_workspace_bytes() (a work list of 16 bytes per block of
 * 128 / (Hq / Hkv) positions and key/value head).
 */
size_t jet_prefill_workspace_bytes(const jet_sizes* n, const jet_dims* dims);
jet_status jet_prefill_attend(const jet_layout* lay, const jet_dims* dims, const void* q,
                              const void* k, const void* v, void* o, void* ws, size_t ws_bytes,
                              void* stream);

/*
 * jet_prefill_state - the prefill of a linear-attention layer: every request's
 * P_r prefix tokens fed in order through the recurrence `rule` (JET_RECUR_*,
 * as for jet_fork_state_rule) starting from s_init.
 *   s_init  [R, Hl, dk, dv] float32   initial states; NULL means zeros
 *   q, k    [total_prefix, Hl, dk] dims.dtype; v [total_prefix, Hl, dv]
 *   alpha, beta [total_prefix, Hl] float32
 *   o       [total_prefix, Hl, dv] dims.dtype  each prefix token's output
 *   s_out   [R, Hl, dk, dv] float32   the state after the prefix: the
 *           s_prefix every candidate forks from (Sec. 4.1)
 * Requests and heads run in parallel. bf16 states of 128 x 128 take the
 * chunked form on the tensor cores (64 tokens at a time, one CTA per
 * request and head; an exact rearrangement of the recurrence with float32-
 * like accuracy); float32 and other state shapes run the tokens one after
 * another (32- or 64-column slices of the state in parallel).
 */
jet_status jet_prefill_state(const jet_layout* lay, const jet_dims* dims, int32_t rule,
                             const float* s_init, const void* q, const void* k, const void* v,
                             const float* alpha, const float* beta, void* o, float* s_out,
                             void* stream);

/*
 * jet_fork_state - per-candidate fork of a linear-attention recurrent state
 * (Sec. 4.1: each candidate continues from the unchanged prefix state).
 *   s_prefix [R, Hl, dk, dv] float32  state after the prefix (read only)
 *   q, k     [F, Hl, dk]  dims.dtype  per fed token; k is expected unit-norm
 *   v        [F, Hl, dv]  dims.dtype
 *   alpha, beta [F, Hl] float32       gates
 *   o        [F, Hl, dv]  dims.dtype  output o_t = S_t^T q_t / sqrt(dk)
 *   s_fork   [C, Hl, dk, dv] float32  state after each candidate's last fed
 *            token (a copy of the prefix state when m_c = 1); may be NULL
 * Each fed token applies S <- alpha (S - beta k (k^T S)) + beta k v^T (gated
 * delta rule; the paper does not name its recurrence). All candidates run
 * concurrently from one read of the prefix state.
 */
jet_status jet_fork_state(const jet_layout* lay, const jet_dims* dims, const float* s_prefix,
                          const void* q, const void* k, const void* v, const float* alpha,
                          const float* beta, void* o, float* s_fork, void* stream);

/*
 * jet_fork_state_rule - jet_fork_state with the recurrence chosen by `rule`:
 * JET_RECUR_DELTA, the gated delta rule above (what jet_fork_state runs), or
 * JET_RECUR_GLA, plain gated linear attention S <- alpha S + beta k v^T (no
 * erase term), with the same inputs, outputs and read-out. Any other rule:
 * JET_ERR_ARG.
 */
jet_status jet_fork_state_rule(const jet_layout* lay, const jet_dims* dims, int32_t rule,
                               const float* s_prefix, const void* q, const void* k, const void* v,
                               const float* alpha, const float* beta, void* o, float* s_fork,
                               void* stream);

/*
 * jet_score_candidates - LM head, full-vocabulary log-softmax and target
 * gather (Eq. 1, Eq. 2), then candidate scores (Eq. 3).
 *   hidden      [N, D]  dims.dtype  LM-head input of every row
 *   w_lm        [V, D]  dims.dtype  LM-head weights (logit z_v = hidden . w_lm[v])
 *   tok_logprob [T] float32         l_{c,t} in candidate order
 *   cand_score  [C] float32         s(c|x) = sum_t l_{c,t}, summed in t order
 * The N x V logits are reduced on chip to per-tile (max, sum of exp) pairs and
 * never written to memory. bf16 inputs use the tensor cores with float32
 * accumulation; float32 inputs use float32 FMA.
 * ws/ws_bytes: scratch of at least jet_workspace_bytes().
 */
jet_status jet_score_candidates(const jet_layout* lay, const jet_dims* dims, const void* hidden,
                                const void* w_lm, float* tok_logprob, float* cand_score,
                                void* ws, size_t ws_bytes, void* stream);

/*
 * jet_evaluate - evaluation against a gold answer (Sec. 3.3, Sec. 5.1).
 *   cand_score [C] float32  s(c|x) (jet_score_candidates)
 *   choice     [R] int32    the chosen candidate of each request (jet_decide)
 *   gold       [C] uint8    nonzero for every candidate whose label carries
 *                           the gold answer text (several labels may)
 *   nll        [R] float32  -log sum_{gold c} q(c), q from Eq. 4: the
 *                           probabilities of equivalent labels are summed;
 *                           +infinity when no candidate of the request is gold
 *   correct    [R] int32    1 when the chosen label carries the gold text
 * For binary requests the choice is the argmax of {false, true}, i.e. q(true)
 * thresholded at 1/2 with a tie going to false. Batch accuracy and mean NLL
 * are the caller's sums over requests.
 */
jet_status jet_evaluate(const jet_layout* lay, const float* cand_score, const int32_t* choice,
                        const uint8_t* gold, float* nll, int32_t* correct, void* stream);

/*
 * Low-precision LM head. The paper runs its models with 8-bit (Q8_0) and
 * 4-bit (Q4_K_M) weights (Appendix A); here a matrix row is stored as OCP FP8
 * E4M3 codes (1 sign, 4 exponent bits with bias 7, 3 mantissa bits; largest
 * finite value 448, no infinities) plus one float32 scale s, with
 * x[k] ~= s * decode(q[k]).
 *
 * jet_quantize_rows_e4m3 - quantise the bf16 matrix x [rows, D] row by row:
 * amax = max_k |x[k]| (float32), s = amax / 448, q[k] = e4m3(x[k] * (448 /
 * amax)) rounded to nearest even and saturated at +-448; a row of zeros gets
 * s = 0 and zero codes. q [rows, D] uint8, scale [rows] float32 (device,
 * caller-owned). Errors: JET_ERR_ARG (rows < 0, null pointer), JET_ERR_SHAPE
 * (D not a positive multiple of 16), JET_ERR_ALIGN. Used once for w_lm (model
 * state); jet_score_candidates_e4m3 applies it to the hidden states itself.
 */
jet_status jet_quantize_rows_e4m3(const void* x, int32_t rows, int32_t D, uint8_t* q, float* scale,
                                  void* stream);

/* Workspace bytes of jet_prefix_attend and jet_score_candidates_e4m3 (the
 * larger of the two). 0 on invalid arguments. */
size_t jet_workspace_bytes_e4m3(const jet_sizes* n, const jet_dims* dims);

/*
 * jet_score_candidates_e4m3 - jet_score_candidates with an e4m3 LM head:
 *   hidden      [N, D] bf16     quantised per row (token) into the workspace
 *   w_q         [V, D] uint8    e4m3 codes of w_lm (jet_quantize_rows_e4m3)
 *   w_scale     [V] float32     their per-row scales
 *   tok_logprob, cand_score     as for jet_score_candidates
 * The logit is z[n, v] = s_h[n] s_w[v] sum_k decode(h_q[n, k]) decode(w_q[v, k]),
 * accumulated in float32 on the tensor cores (tcgen05 kind::f8f6f4); the
 * log-softmax, gather and candidate sums are those of jet_score_candidates.
 * dims.dtype must be JET_DTYPE_BF16 (else JET_ERR_UNSUPPORTED) and dims.D a
 * multiple of 16 (else JET_ERR_SHAPE). ws/ws_bytes: scratch of at least
 * jet_workspace_bytes_e4m3().
 */
jet_status jet_score_candidates_e4m3(const jet_layout* lay, const jet_dims* dims,
                                     const void* hidden, const uint8_t* w_q, const float* w_scale,
                                     float* tok_logprob, float* cand_score, void* ws,
                                     size_t ws_bytes, void* stream);

/*
 * 4-bit LM head (w4; the analogue of the paper's 4-bit weights, Appendix A,
 * whose codes come in 32-element blocks with their own scales). A row x of
 * w_lm is stored as OCP FP4 E2M1 codes (1 sign, 2 exponent bits with bias 1,
 * 1 mantissa bit: magnitudes 0, .5, 1, 1.5, 2, 3, 4, 6), one power-of-two
 * exponent e in [-5, 0] per 32-element block and one float32 scale s per row,
 * with x[k] ~= s * 2^e(k / 32) * value(code[k]):
 *   amax = max |x|, s = amax / 6, inv = 6 / amax (float32, rounded to nearest);
 *   block b: t = (max |x| over the block) * inv, e = the smallest integer in
 *   [-5, 0] with t <= 6 * 2^e (0 if none); code = e2m1(x * (inv * 2^-e)),
 *   nearest with ties to the even code, saturated at +-6. A row of zeros gets
 *   s = 0, zero codes and e = -5.
 *
 * Layout of the w4 buffer (what the block-scaled tensor-core path reads):
 * with Vp = 128 ceil(V / 128) rows and Kp = 128 ceil(D / 128) codes per row,
 *   - a code region of Vp * Kp / 2 bytes, row-major: code k of row v is the
 *     nibble (k & 1) of byte v * Kp / 2 + k / 2 (element 2 j in the low nibble
 *     of byte j), in the OCP E2M1 encoding (sign in bit 3);
 *   - then a scale-factor region of one 512-byte chunk per (vocabulary tile vt
 *     of 128 rows, K slice kb of 128 codes), chunk index vt ceil(D / 128) + kb:
 *     byte 16 i + 4 j + c of a chunk is the UE8M0 factor 127 + e of block c of
 *     the slice in row 32 j + i of the tile (the order in which one tcgen05.cp
 *     of 32 x 128 bits places the chunk in tensor memory for the block-scaled
 *     MMA). Rows past V and codes past D are zero codes; their blocks have
 *     e = -5.
 */

/* Bytes of the w4 buffer of a [V, D] matrix (codes and scale factors):
 * ceil(V / 128) * ceil(D / 128) * (8192 + 512); 0 on invalid arguments. */
size_t jet_w4_bytes(int64_t V, int64_t D);

/*
 * jet_quantize_w4 - quantise the bf16 matrix w [V, D] (device, row-major) into
 * w4 (jet_w4_bytes(V, D) bytes, 16-byte aligned) and scale [V] float32.
 * Errors: JET_ERR_ARG (V < 1 or a null pointer), JET_ERR_SHAPE (D not a
 * positive multiple of 16), JET_ERR_ALIGN. Done once per model (w_lm is model
 * state).
 */
jet_status jet_quantize_w4(const void* w, int64_t V, int64_t D, uint8_t* w4, float* scale,
                           void* stream);

/*
 * jet_score_candidates_w4 - jet_score_candidates with a 4-bit LM head:
 *   hidden      [N, D] bf16     quantised per row (token) to e4m3 into the
 *                               workspace, as in jet_score_candidates_e4m3
 *   w4          codes and scale factors of w_lm from jet_quantize_w4 with the
 *               same V, D (32-byte aligned, else JET_ERR_ALIGN)
 *   w_scale     [V] float32     their per-row scales
 * The logit is z[n, v] = s_h[n] s_w[v] sum_k decode(h_q[n, k]) 2^e value(code),
 * accumulated in float32 on the tensor cores by the block-scaled MMA (E2M1
 * weight codes with one UE8M0 factor 2^e per 32-element block, e4m3 hidden
 * codes: every product is exact); log-softmax, gather and sums as in
 * jet_score_candidates. dims as for jet_score_candidates_e4m3; workspace
 * jet_workspace_bytes_e4m3().
 */
jet_status jet_score_candidates_w4(const jet_layout* lay, const jet_dims* dims,
                                   const void* hidden, const uint8_t* w4, const float* w_scale,
                                   float* tok_logprob, float* cand_score, void* ws,
                                   size_t ws_bytes, void* stream);

/*
 * MXFP8 LM head (the microscaling form of the paper's 8-bit weights, Appendix
 * A: 8-bit codes in 32-element blocks that each carry a scale). Every row of
 * the weights and of the hidden states is cut into 32-element blocks (the last
 * may be shorter); block b gets the shared exponent
 *   X = floor(log2(max |x| over the block)) - 8, clamped to [-127, 127]
 *   (-127 for a block of zeros or of subnormal maxima),
 * stored as the UE8M0 byte X + 127, and its elements the OCP FP8 E4M3 codes of
 * x * 2^-X (nearest, ties to even, saturating at +-448). The value of a code
 * is 2^X decode(code); there is no further per-row scale.
 *
 * Layout of an MXFP8 weight buffer for [V, D] (jet_mxfp8_bytes(V, D) bytes):
 *   - codes [V, D] row-major (V D bytes, rounded up to 256);
 *   - then one 512-byte chunk of scale factors per (vocabulary tile vt of 128
 *     rows, K slice kb of 128 elements), chunk vt ceil(D / 128) + kb, byte
 *     16 i + 4 j + c holding block c of the slice of row 128 vt + 32 j + i
 *     (127 for rows past V).
 */
size_t jet_mxfp8_bytes(int64_t V, int64_t D);

/*
 * jet_quantize_mxfp8 - quantise the bf16 matrix w [V, D] (device, row-major)
 * into `out` (jet_mxfp8_bytes(V, D) bytes, 16-byte aligned). Errors:
 * JET_ERR_ARG, JET_ERR_SHAPE (D not a positive multiple of 16), JET_ERR_ALIGN.
 * Done once per model.
 */
jet_status jet_quantize_mxfp8(const void* w, int64_t V, int64_t D, uint8_t* out, void* stream);

/* Workspace bytes of jet_score_candidates_mxfp8 (the bf16 path's, the hidden
 * states' codes and their scale factors); 0 on invalid arguments. */
size_t jet_workspace_bytes_mxfp8(const jet_sizes* n, const jet_dims* dims);

/*
 * jet_score_candidates_mxfp8 - jet_score_candidates with an MXFP8 LM head:
 *   hidden      [N, D] bf16     quantised to MXFP8 into the workspace
 *   w_mx        the weights from jet_quantize_mxfp8 with the same V, D
 * The logit is z[n, v] = sum_b 2^(X_h[n, b] + X_w[v, b]) sum_{k in b}
 * decode(h_q[n, k]) decode(w_q[v, k]), accumulated in float32 on the tensor
 * cores by the block-scaled MMA (both sets of scale factors applied by the
 * hardware); log-softmax, gather and sums as in jet_score_candidates. dims:
 * dtype JET_DTYPE_BF16, D a positive multiple of 16; workspace
 * jet_workspace_bytes_mxfp8().
 */
jet_status jet_score_candidates_mxfp8(const jet_layout* lay, const jet_dims* dims,
                                      const void* hidden, const uint8_t* w_mx,
                                      float* tok_logprob, float* cand_score, void* ws,
                                      size_t ws_bytes, void* stream);

/*
 * Hybrid decoder stacks (Sec. 4.1: hybrid models keep a recurrent state per
 * linear-attention layer, restored for every candidate, and reuse the prefix
 * cache at attention layers). jet_stack_forward runs L pre-norm decoder
 * layers over the step's N rows - each request's shared row and its
 * candidates' fed tokens - with a fork of the recurrent state at every
 * linear-attention layer:
 *   h  = RMSNorm(x) * g1                          (eps 1e-6)
 *   full layer:   q, k, v = h w_mix^T; the step's cascade attention over the
 *                 layer's prefix keys/values plus each candidate's own fed
 *                 tokens (jet_prefix_attend); the shared row's own key/value
 *                 is the prefix's last position
 *   linear layer: q, k, v, a, b = h w_mix^T; k normalised per head;
 *                 alpha = sigmoid(a), beta = sigmoid(b); the fed tokens run
 *                 the recurrence from the layer's prefix state
 *                 (jet_fork_state_rule, stack.rule); a shared row reads the
 *                 prefix state: o = S_prefix^T q / sqrt(dk)
 *   x  = x + o w_o^T
 *   x  = x + (SiLU(RMSNorm(x) * g2 w_gate^T) * (... w_up^T)) w_down^T
 * Activations are bf16 between operations (f32 inside each); the
 * projections run on the tensor cores.
 */
enum { JET_LAYER_LINEAR = 0, JET_LAYER_FULL = 1 };

typedef struct jet_stack_layer {
  int32_t kind;        /* JET_LAYER_LINEAR or JET_LAYER_FULL                     */
  int32_t reserved;
  const void* g1;      /* [D] bf16 RMSNorm gains before the mixer                */
  const void* g2;      /* [D] bf16 RMSNorm gains before the MLP                  */
  const void* w_mix;   /* bf16; full: [(Hq + 2 Hkv) d, D], rows q heads, k heads,
                          v heads; linear: [Hl (2 dk + dv) + 2 Hl, D], rows q, k,
                          v heads, then the Hl decay and Hl write-strength logits */
  const void* w_o;     /* bf16 [D, Hq d] (full) or [D, Hl dv] (linear)           */
  const void* w_gu;    /* bf16 [2 Dff, D]: rows 128 t .. + 63 are the gate rows of
                          features 64 t .. + 63, rows 128 t + 64 .. + 127 their
                          up rows                                                */
  const void* w_d;     /* bf16 [D, Dff]                                           */
  const void* k_pre;   /* full: bf16 [sum P, Hkv, d] prefix keys; linear: NULL    */
  const void* v_pre;   /* full: bf16 [sum P, Hkv, d] prefix values               */
  const float* s_prefix; /* linear: [R, Hl, dk, dv] prefix states; full: NULL   */
} jet_stack_layer;

typedef struct jet_stack {
  int32_t L;           /* layers                                                  */
  int32_t Dff;         /* MLP width, a positive multiple of 64                    */
  int32_t rule;        /* JET_RECUR_* of the linear layers                        */
  int32_t reserved;
  const jet_stack_layer* layers; /* host array of L layers, read during the call */
} jet_stack;

/* Workspace bytes of jet_stack_forward for these sizes, dims and MLP width;
 * 0 on invalid arguments. */
size_t jet_stack_workspace_bytes(const jet_sizes* n, const jet_dims* dims, int32_t Dff);

/*
 * jet_stack_forward - x = the stack applied to x0 (both [N, D] bf16, device;
 * x may equal x0). dims: dtype JET_DTYPE_BF16, D a multiple of 16; with a
 * full layer Hq, Hkv, d as for jet_prefix_attend; with a linear layer Hl even,
 * dk = 128, dv a multiple of 32. The result is the hidden state that
 * jet_score_candidates takes. Errors: as for the calls it makes, plus
 * JET_ERR_ARG (a null layer pointer, an unknown kind or rule, L < 0),
 * JET_ERR_SHAPE (Dff), JET_ERR_WORKSPACE.
 */
jet_status jet_stack_forward(const jet_layout* lay, const jet_dims* dims, const jet_stack* stack,
                             const void* x0, void* x, void* ws, size_t ws_bytes, void* stream);

/*
 * jet_score_candidates_noalloc - jet_score_candidates without caller-owned
 * scratch memory. The paper has no counterpart to this entry point: it exists
 * for callers that cannot call cudaMalloc, such as a host application that
 * owns every device allocation and passes its plug-ins only the tensors they
 * work on, or a serving loop that must not allocate (cudaMalloc can
 * synchronise the device and can fail under memory pressure) once it runs.
 * Arguments and results are those of jet_score_candidates minus ws/ws_bytes.
 * - Scratch is a fixed 16 MiB array inside the library (a __device__ array that
 *   every GPU loading the library holds until the process exits). A batch
 *   needs N * ceil(V / 128) * 8 + T * 4 + N * 4 bytes (each term rounded up to
 *   256); larger batches get JET_ERR_CAPACITY and nothing is launched. With
 *   V = 151,936 that allows about 1,700 rows.
 * - The call allocates nothing and calls no allocating library routine.
 * - The first call on each device looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current); make that first call
 *   before any stream capture on the device.
 * - Every call shares the one array: calls whose work overlaps on the GPU
 *   (other streams, other threads) race on it and must be ordered by the
 *   caller. No part of the array needs clearing between calls: each element a
 *   call reads is written earlier by the same call.
 */
jet_status jet_score_candidates_noalloc(const jet_layout* lay, const jet_dims* dims,
                                        const void* hidden, const void* w_lm,
                                        float* tok_logprob, float* cand_score, void* stream);

/*
 * jet_decide - decision rules (Eq. 4, Eq. 5, Sec. 3.3).
 *   cand_score [C] float32   s(c|x)
 *   q          [C] float32   q(c) = exp(s_c - M) / sum_d exp(s_d - M), M = max s
 *   choice     [R] int32     argmax_c s_c, ties to the lowest candidate index
 *   value      [R] float32   ARGMAX: q(choice); BINARY: q(true) = q of
 *                            candidate 1 (the set is {false, true}, every
 *                            request needs C_r = 2, else JET_ERR_SHAPE);
 *                            ORDINAL: sum_i i q(i), zero-based levels
 */
jet_status jet_decide(const jet_layout* lay, int32_t mode, const float* cand_score, float* q,
                      int32_t* choice, float* value, void* stream);

/*
 * jet_device_status - wait for `stream`, then report and clear the current
 * device's status word: JET_OK, JET_ERR_DEVICE (a kernel skipped an
 * out-of-range layout index) or JET_ERR_TIMEOUT (a bounded wait gave up).
 * A failed CUDA call returns JET_ERR_CUDA.
 */
jet_status jet_device_status(void* stream, jet_status* out);

/*
 * jet_set_wait_budget_ns - budget of one bounded wait inside the tensor-core
 * kernels (the attention, LM-head and projection kernels poll mbarriers
 * between their roles). A wait that runs past it gives up: the kernel stops
 * issuing work, lets the copies and tensor-core operations it already issued
 * finish, frees its tensor memory, returns, and the next jet_device_status
 * reports JET_ERR_TIMEOUT. 0 restores the default of 2 s. The value is read
 * when an entry point launches a kernel, so it applies to later calls only;
 * it is process-wide (all devices and threads). A short budget is how a
 * caller (or a test) checks the timeout path without a stalled GPU.
 * Returns the budget that was in force before the call.
 */
uint64_t jet_set_wait_budget_ns(uint64_t ns);

/*
 * jet_set_test_stall - test hook for the timeout path. While `on` is nonzero,
 * every tensor-core kernel launched afterwards withholds its first load (the
 * LM head and the projections their first operand stage, the attention its
 * first query block), so that the role waiting for it waits for something
 * nothing will provide: that wait runs out its budget (jet_set_wait_budget_ns)
 * and the kernel ends as described there, reporting JET_ERR_TIMEOUT. Results
 * of such calls are meaningless. Process-wide, read at launch; returns the
 * previous setting. Off unless set.
 */
int32_t jet_set_test_stall(int32_t on);

/*
 * jet_launch_count - kernels this library has launched in this process so
 * far (every successful launch by any entry point, on any device or thread).
 * The difference across a region is the number of kernels it launched.
 */
uint64_t jet_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* JET_H */
