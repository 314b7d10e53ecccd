// Refusal-prefix trie shared by the gate kernels and the fused sample head:
// the library-owned trie object, its device view, and one probe token through
// the hard gate (the compatibility predicate C of Sec. 3 on a token trie, and
// the outcome of Alg. 1), with the row mask that follows from a gate state.
// While q is a path of the trie it is a prefix of some refusal prefix; once q
// reaches a node that ends a prefix of length >= min_confirm (the two-token
// minimum of App. D) every extension stays compatible; leaving the trie before
// that is incompatible.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "rgd.h"

struct rgd_trie {
  int32_t num_nodes = 0;
  int32_t num_edges = 0;
  int32_t* child_begin = nullptr;  // [num_nodes + 1]
  int32_t* child_tok = nullptr;    // [num_edges], sorted within a node
  int32_t* child_node = nullptr;   // [num_edges]
  uint8_t* confirm = nullptr;      // [num_nodes]: ends a prefix of length >= min_confirm
  int32_t max_children = 0;        // the largest number of children of a node
  int device = 0;
};

namespace rgd {
namespace {

struct TrieView {
  const int32_t* child_begin;
  const int32_t* child_tok;
  const int32_t* child_node;
  const uint8_t* confirm;
};

// Index of `tok` among the children of `node`, or -1.
__device__ __forceinline__ int32_t find_child(const TrieView& t, int32_t node, int32_t tok) {
  int32_t lo = __ldg(t.child_begin + node), hi = __ldg(t.child_begin + node + 1);
  while (lo < hi) {
    const int32_t mid = (lo + hi) >> 1;
    const int32_t v = __ldg(t.child_tok + mid);
    if (v < tok) lo = mid + 1;
    else hi = mid;
  }
  if (lo < __ldg(t.child_begin + node + 1) && __ldg(t.child_tok + lo) == tok) return lo;
  return -1;
}

// One probe token y (the stop token, or y >= 0) through the hard gate, for a
// state whose probe has not ended.  child(y) gives the trie edge labelled y
// out of s.node as {node it leads to, whether that node confirms}, or
// {-1, 0} when there is none.
template <typename Child>
__device__ void consume_token_with(rgd_gate_state& s, int32_t y, int32_t eos, int32_t max_len,
                                   bool root_has_children, Child&& child) {
  if (eos >= 0 && y == eos) {
    const int32_t step = s.steps++;
    s.done = 1;
    if (s.decision == RGD_PENDING) {
      // a pending probe is compatible, except the empty probe against an empty set
      const bool ok = s.length > 0 || root_has_children;
      s.decision = ok ? RGD_REFUSAL : RGD_NON_REFUSAL;
      s.decisive_step = step;
    }
    return;
  }
  const int32_t step = s.steps++;
  s.length++;
  if (!s.confirmed) {
    const int2 e = child(y);
    if (e.x < 0) {
      s.decision = RGD_NON_REFUSAL;
      s.decisive_step = step;
      s.done = 1;
      return;
    }
    s.node = e.x;
    if (e.y) {
      s.confirmed = 1;
      if (s.decision == RGD_PENDING) {
        s.decision = RGD_REFUSAL;
        s.decisive_step = step;
      }
    }
  }
  if (s.length >= max_len) {
    s.done = 1;
    if (s.decision == RGD_PENDING) {
      s.decision = RGD_REFUSAL;
      s.decisive_step = step;
    }
  }
}

// consume_token_with, the edge looked up in the trie.
__device__ __forceinline__ void consume_token(const TrieView& t, rgd_gate_state& s, int32_t y, int32_t eos,
                                              int32_t max_len, bool root_has_children) {
  consume_token_with(s, y, eos, max_len, root_has_children, [&](int32_t tok) {
    const int32_t e = find_child(t, s.node, tok);
    if (e < 0) return make_int2(-1, 0);
    const int32_t nd = __ldg(t.child_node + e);
    return make_int2(nd, (int)__ldg(t.confirm + nd));
  });
}

// The gate's row mask: the probe row off once the probe has ended, the sample
// rows off once the outcome is REFUSAL.
__device__ __forceinline__ void mask_rows(const rgd_gate_state& s, uint8_t* row_active, int32_t g,
                                          int32_t rows_per_group) {
  if (!row_active) return;
  uint8_t* ra = row_active + (int64_t)g * rows_per_group;
  if (s.done) ra[0] = 0;
  if (s.decision == RGD_REFUSAL)
    for (int32_t i = 1; i < rows_per_group; ++i) ra[i] = 0;
}

}  // namespace
}  // namespace rgd
