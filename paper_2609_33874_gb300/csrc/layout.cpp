// Host-side construction of the teacher-forced candidate layout.
//
// The layout maps the problem statement (context x with P_r prefix tokens,
// candidates y_c of m_c tokens, Sec. 3.1) to query rows and targets:
// request r's first row is its last prefix position and predicts y_{c,1} for
// every candidate (Sec. 4.1); the row fed with y_{c,t} predicts y_{c,t+1}
// (Eq. 1 conditions z_{c,t,.} on (x, y_{c,<t})). Pure host code: no CUDA call.
#include <algorithm>
#include <climits>
#include <cstring>
#include <vector>

#include "jet.h"

namespace {

inline size_t pad4(size_t x) { return (x + 3) & ~size_t(3); }

// word offsets of the 12 arrays, plus the total, in the order of jet_layout
void word_offsets(const jet_sizes& n, size_t off[14]) {
  const size_t R = size_t(n.R), C = size_t(n.C), N = size_t(n.N), T = size_t(n.T);
  const size_t len[13] = {R + 1, R + 1, R + 1, C + 1, C + 1, T, T, N, N, N, N + 1, T, R};
  size_t o = 0;
  for (int i = 0; i < 13; ++i) {
    off[i] = o;
    o += pad4(len[i]);
  }
  off[13] = o;
}

}  // namespace

extern "C" jet_status jet_layout_plan(int32_t R, const int32_t* prefix_len, const int32_t* n_cand,
                                      const int32_t* cand_len, int32_t V, jet_sizes* out) {
  if (!out || R < 0 || V < 1) return JET_ERR_ARG;
  if (R > 0 && (!prefix_len || !n_cand || !cand_len)) return JET_ERR_ARG;
  long long C = 0, N = 0, T = 0, P = 0;
  int32_t max_prefix = 0, min_cand = INT32_MAX, max_cand = 0, max_rows = 0, max_len = 0;
  for (int32_t r = 0; r < R; ++r) {
    if (prefix_len[r] < 1 || n_cand[r] < 1) return JET_ERR_SHAPE;
    P += prefix_len[r];
    if (prefix_len[r] > max_prefix) max_prefix = prefix_len[r];
    if (n_cand[r] < min_cand) min_cand = n_cand[r];
    if (n_cand[r] > max_cand) max_cand = n_cand[r];
    long long rows = 1;
    for (int32_t i = 0; i < n_cand[r]; ++i) {
      const int32_t m = cand_len[C + i];
      if (m < 1) return JET_ERR_SHAPE;
      rows += m - 1;
      T += m;
      if (m > max_len) max_len = m;
    }
    C += n_cand[r];
    N += rows;
    if (rows > max_rows) max_rows = int32_t(rows);
    if (C > INT32_MAX / 2 || N > INT32_MAX / 2 || T > INT32_MAX / 2 || P > INT32_MAX / 2)
      return JET_ERR_CAPACITY;
  }
  std::memset(out, 0, sizeof(*out));
  out->R = R;
  out->C = int32_t(C);
  out->N = int32_t(N);
  out->T = int32_t(T);
  out->V = V;
  out->total_prefix = int32_t(P);
  out->max_prefix = max_prefix;
  out->min_cand = R > 0 ? min_cand : 0;
  out->max_cand = max_cand;
  out->max_rows = max_rows;
  out->max_len = max_len;
  return JET_OK;
}

extern "C" size_t jet_layout_words(const jet_sizes* n) {
  if (!n || n->R < 0 || n->C < 0 || n->N < 0 || n->T < 0) return 0;
  size_t off[14];
  word_offsets(*n, off);
  return off[13];
}

extern "C" jet_status jet_layout_bind(const jet_sizes* n, const int32_t* words, jet_layout* out) {
  if (!n || !out || (!words && jet_layout_words(n) > 0)) return JET_ERR_ARG;
  if (n->R < 0 || n->C < 0 || n->N < 0 || n->T < 0) return JET_ERR_SHAPE;
  size_t off[14];
  word_offsets(*n, off);
  out->n = *n;
  const int32_t** slots[13] = {&out->prefix_offset, &out->cand_offset,  &out->row_offset,
                               &out->cand_row_offset, &out->tgt_offset, &out->target_ids,
                               &out->tgt_row,       &out->row_req,      &out->row_cand,
                               &out->row_pos,       &out->row_tgt_offset, &out->row_tgt_index,
                               &out->req_order};
  for (int i = 0; i < 13; ++i) *slots[i] = words + off[i];
  return JET_OK;
}

extern "C" jet_status jet_layout_build(int32_t R, const int32_t* prefix_len, const int32_t* n_cand,
                                       const int32_t* cand_len, const int32_t* target_ids, int32_t V,
                                       int32_t* words, size_t n_words, jet_layout* out) {
  if (!out) return JET_ERR_ARG;
  jet_sizes n;
  jet_status st = jet_layout_plan(R, prefix_len, n_cand, cand_len, V, &n);
  if (st != JET_OK) return st;
  if (n.T > 0 && !target_ids) return JET_ERR_ARG;
  for (int32_t j = 0; j < n.T; ++j)
    if (target_ids[j] < 0 || target_ids[j] >= V) return JET_ERR_RANGE;
  const size_t need = jet_layout_words(&n);
  if (need > 0 && (!words || n_words < need)) return JET_ERR_WORKSPACE;
  std::memset(words, 0, need * sizeof(int32_t));
  jet_layout_bind(&n, words, out);
  size_t off[14];
  word_offsets(n, off);
  int32_t* prefix_offset = words + off[0];
  int32_t* cand_offset = words + off[1];
  int32_t* row_offset = words + off[2];
  int32_t* cand_row_offset = words + off[3];
  int32_t* tgt_offset = words + off[4];
  int32_t* tids = words + off[5];
  int32_t* tgt_row = words + off[6];
  int32_t* row_req = words + off[7];
  int32_t* row_cand = words + off[8];
  int32_t* row_pos = words + off[9];
  int32_t* row_tgt_offset = words + off[10];
  int32_t* row_tgt_index = words + off[11];
  int32_t* req_order = words + off[12];

  int32_t row = 0, c = 0, j = 0;
  prefix_offset[0] = 0;
  cand_offset[0] = 0;
  for (int32_t r = 0; r < R; ++r) {
    prefix_offset[r + 1] = prefix_offset[r] + prefix_len[r];
    cand_offset[r + 1] = cand_offset[r] + n_cand[r];
    const int32_t shared = row;
    row_offset[r] = shared;
    row_req[row] = r;
    row_cand[row] = -1;
    row_pos[row] = 0;
    ++row;
    for (int32_t i = 0; i < n_cand[r]; ++i, ++c) {
      const int32_t m = cand_len[c];
      const int32_t first = row;
      cand_row_offset[c] = first;
      for (int32_t t = 1; t < m; ++t, ++row) {  // rows fed with y_{c,1..m-1}
        row_req[row] = r;
        row_cand[row] = c;
        row_pos[row] = t;
      }
      tgt_offset[c] = j;
      for (int32_t t = 1; t <= m; ++t, ++j) {   // targets y_{c,1..m}
        tids[j] = target_ids[j];
        tgt_row[j] = (t == 1) ? shared : first + (t - 2);
      }
    }
  }
  row_offset[R] = row;
  cand_row_offset[n.C] = row;
  tgt_offset[n.C] = j;

  // group targets by predicting row (counting sort; stable in target index)
  std::vector<int32_t> count(size_t(n.N) + 1, 0);
  for (int32_t t = 0; t < n.T; ++t) ++count[size_t(tgt_row[t]) + 1];
  row_tgt_offset[0] = 0;
  for (int32_t r = 0; r < n.N; ++r) row_tgt_offset[r + 1] = row_tgt_offset[r] + count[size_t(r) + 1];
  std::vector<int32_t> fill(row_tgt_offset, row_tgt_offset + n.N);
  for (int32_t t = 0; t < n.T; ++t) row_tgt_index[fill[size_t(tgt_row[t])]++] = t;

  // requests by decreasing prefix length (ties: lower index first); kernels
  // hand out long prefixes first so that their work balances across SMs
  for (int32_t r = 0; r < R; ++r) req_order[r] = r;
  std::stable_sort(req_order, req_order + R,
                   [&](int32_t x, int32_t y) { return prefix_len[x] > prefix_len[y]; });
  return JET_OK;
}
