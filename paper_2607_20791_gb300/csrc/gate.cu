// Refusal-prefix gate: host-built token trie + per-token hard-gate kernel.
//
// The compatibility predicate C(q, P) of Sec. 3 holds when q is a prefix of some
// refusal prefix pi, or some pi (with |pi| >= min_confirm, the two-token minimum
// of App. D) is a prefix of q.  On a trie of P this becomes a walk: while q is a
// trie path it is a prefix of some pi; once q reaches a node that ends a pi of
// length >= min_confirm ("confirmed") every extension stays compatible; leaving
// the trie before that is incompatible.  The hard gate of Alg. 1 applies the
// predicate after every greedy probe token (the cap c does not change the
// outcome of the hard gate).
#include <algorithm>
#include <map>
#include <vector>

#include "common.h"
#include "ptx.cuh"

struct rgd_trie {
  int32_t num_nodes = 0;
  int32_t num_edges = 0;
  int32_t* child_begin = nullptr;  // [num_nodes + 1]
  int32_t* child_tok = nullptr;    // [num_edges], sorted within a node
  int32_t* child_node = nullptr;   // [num_edges]
  uint8_t* confirm = nullptr;      // [num_nodes]: ends a prefix of length >= min_confirm
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

__global__ void gate_state_init_kernel(rgd_gate_state* st, int32_t groups) {
  const int32_t g = blockIdx.x * blockDim.x + threadIdx.x;
  if (g >= groups) return;
  rgd_gate_state s;
  s.node = 0;
  s.length = 0;
  s.steps = 0;
  s.decisive_step = -1;
  s.decision = RGD_PENDING;
  s.confirmed = 0;
  s.done = 0;
  s.reserved = 0;
  st[g] = s;
}

__global__ void probe_gate_kernel(TrieView t, int32_t groups, int32_t rows_per_group,
                                  const int32_t* __restrict__ tokens, int32_t n_tokens, int64_t stride,
                                  int32_t eos, int32_t max_len, rgd_gate_state* __restrict__ state,
                                  uint8_t* __restrict__ row_active, int32_t* dev_status) {
  const int32_t g = blockIdx.x * blockDim.x + threadIdx.x;
  if (g >= groups) return;
  rgd_gate_state s = state[g];
  const bool root_has_children = __ldg(t.child_begin + 1) > __ldg(t.child_begin);
  bool bad_token = false;
  for (int32_t k = 0; k < n_tokens && !s.done; ++k) {
    const int32_t y = __ldg(tokens + (int64_t)g * stride + k);
    if (eos >= 0 && y == eos) {
      const int32_t step = s.steps++;
      s.done = 1;
      if (s.decision == RGD_PENDING) {
        // a pending probe is compatible, except the empty probe against an empty set
        const bool ok = s.length > 0 || root_has_children;
        s.decision = ok ? RGD_REFUSAL : RGD_NON_REFUSAL;
        s.decisive_step = step;
      }
      break;
    }
    if (y < 0) {
      bad_token = true;
      continue;
    }
    const int32_t step = s.steps++;
    s.length++;
    if (!s.confirmed) {
      const int32_t e = find_child(t, s.node, y);
      if (e < 0) {
        s.decision = RGD_NON_REFUSAL;
        s.decisive_step = step;
        s.done = 1;
        break;
      }
      s.node = __ldg(t.child_node + e);
      if (__ldg(t.confirm + s.node)) {
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
  state[g] = s;
  if (bad_token && dev_status) atomicOr(dev_status, RGD_DEV_BAD_TOKEN);
  if (row_active) {
    uint8_t* ra = row_active + (int64_t)g * rows_per_group;
    if (s.done) ra[0] = 0;
    if (s.decision == RGD_REFUSAL)
      for (int32_t i = 1; i < rows_per_group; ++i) ra[i] = 0;
  }
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" int rgd_trie_create(const int32_t* tokens, const int64_t* offsets, int32_t n_seq,
                               int32_t min_confirm, rgd_trie** out) {
  clear_error();
  RGD_CHECK_ARG(out != nullptr, "rgd_trie_create: out is NULL");
  *out = nullptr;
  RGD_CHECK_ARG(n_seq >= 0, "rgd_trie_create: n_seq < 0");
  RGD_CHECK_ARG(min_confirm >= 1, "rgd_trie_create: min_confirm must be >= 1");
  RGD_CHECK_ARG(n_seq == 0 || (tokens != nullptr && offsets != nullptr),
                "rgd_trie_create: tokens/offsets are NULL");
  if (n_seq > 0) RGD_CHECK_ARG(offsets[0] == 0, "rgd_trie_create: offsets[0] != 0");
  // host build: nodes with ordered children (std::map keeps tokens sorted)
  std::vector<std::map<int32_t, int32_t>> kids(1);
  std::vector<int32_t> depth(1, 0);
  std::vector<uint8_t> terminal(1, 0);
  for (int32_t s = 0; s < n_seq; ++s) {
    const int64_t b = offsets[s], e = offsets[s + 1];
    RGD_CHECK_ARG(e > b, "rgd_trie_create: sequence %d is empty or offsets decrease", s);
    int32_t node = 0;
    for (int64_t i = b; i < e; ++i) {
      const int32_t tok = tokens[i];
      RGD_CHECK_ARG(tok >= 0, "rgd_trie_create: negative token in sequence %d", s);
      auto it = kids[node].find(tok);
      if (it == kids[node].end()) {
        const int32_t nn = (int32_t)kids.size();
        kids[node][tok] = nn;
        kids.emplace_back();
        depth.push_back(depth[node] + 1);
        terminal.push_back(0);
        node = nn;
      } else {
        node = it->second;
      }
    }
    terminal[node] = 1;
  }
  const int32_t nn = (int32_t)kids.size();
  std::vector<int32_t> begin(nn + 1, 0), ctok, cnode;
  std::vector<uint8_t> confirm(nn, 0);
  for (int32_t n = 0; n < nn; ++n) {
    begin[n] = (int32_t)ctok.size();
    for (const auto& kv : kids[n]) {
      ctok.push_back(kv.first);
      cnode.push_back(kv.second);
    }
    confirm[n] = (terminal[n] && depth[n] >= min_confirm) ? 1 : 0;
  }
  begin[nn] = (int32_t)ctok.size();
  if (ctok.empty()) {  // keep device arrays non-empty
    ctok.push_back(-1);
    cnode.push_back(0);
  }
  rgd_trie* t = new rgd_trie();
  t->num_nodes = nn;
  t->num_edges = begin[nn];
  cudaGetDevice(&t->device);
  cudaError_t err = cudaSuccess;
  auto upload = [&](void** dst, const void* src, size_t bytes) {
    if (err != cudaSuccess) return;
    err = cudaMalloc(dst, bytes);
    if (err == cudaSuccess) err = cudaMemcpy(*dst, src, bytes, cudaMemcpyHostToDevice);
  };
  upload((void**)&t->child_begin, begin.data(), begin.size() * sizeof(int32_t));
  upload((void**)&t->child_tok, ctok.data(), ctok.size() * sizeof(int32_t));
  upload((void**)&t->child_node, cnode.data(), cnode.size() * sizeof(int32_t));
  upload((void**)&t->confirm, confirm.data(), confirm.size());
  if (err != cudaSuccess) {
    rgd_trie_destroy(t);
    return cuda_error(err, "rgd_trie_create upload");
  }
  *out = t;
  return RGD_OK;
}

extern "C" int rgd_trie_destroy(rgd_trie* t) {
  if (!t) return RGD_OK;
  cudaFree(t->child_begin);
  cudaFree(t->child_tok);
  cudaFree(t->child_node);
  cudaFree(t->confirm);
  delete t;
  return RGD_OK;
}

extern "C" int rgd_trie_info(const rgd_trie* t, int32_t* num_nodes, int32_t* num_edges) {
  clear_error();
  RGD_CHECK_ARG(t != nullptr, "rgd_trie_info: trie is NULL");
  if (num_nodes) *num_nodes = t->num_nodes;
  if (num_edges) *num_edges = t->num_edges;
  return RGD_OK;
}

extern "C" int rgd_gate_state_init(rgd_gate_state* state, int32_t groups, rgd_stream_t stream) {
  clear_error();
  RGD_CHECK_ARG(groups >= 0, "rgd_gate_state_init: groups < 0");
  if (groups == 0) return RGD_OK;
  RGD_CHECK_ARG(state != nullptr, "rgd_gate_state_init: state is NULL");
  const int threads = 128;
  gate_state_init_kernel<<<(groups + threads - 1) / threads, threads, 0, (cudaStream_t)stream>>>(state, groups);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "gate_state_init launch");
}

extern "C" int rgd_probe_gate(const rgd_trie* trie, int32_t groups, int32_t rows_per_group,
                              const int32_t* probe_tokens, int32_t n_tokens, int64_t token_stride,
                              int32_t eos_token, int32_t max_len, rgd_gate_state* state,
                              uint8_t* row_active, int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  RGD_CHECK_ARG(trie != nullptr, "rgd_probe_gate: trie is NULL");
  RGD_CHECK_ARG(groups >= 0 && rows_per_group >= 1, "rgd_probe_gate: bad groups/rows_per_group");
  RGD_CHECK_ARG(n_tokens >= 0 && token_stride >= n_tokens, "rgd_probe_gate: bad n_tokens/token_stride");
  RGD_CHECK_ARG(max_len >= 1, "rgd_probe_gate: max_len must be >= 1");
  if (groups == 0 || n_tokens == 0) return RGD_OK;
  RGD_CHECK_ARG(probe_tokens != nullptr && state != nullptr, "rgd_probe_gate: tokens/state NULL");
  TrieView v{trie->child_begin, trie->child_tok, trie->child_node, trie->confirm};
  const int threads = 128;
  probe_gate_kernel<<<(groups + threads - 1) / threads, threads, 0, (cudaStream_t)stream>>>(
      v, groups, rows_per_group, probe_tokens, n_tokens, token_stride, eos_token, max_len, state, row_active,
      dev_status);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "probe_gate launch");
}
