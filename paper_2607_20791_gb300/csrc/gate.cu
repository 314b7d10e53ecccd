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
#include <cmath>
#include <map>
#include <vector>

#include "common.h"
#include "ptx.cuh"
#include "trie.cuh"

namespace rgd {
namespace {

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
    if (y < 0 && !(eos >= 0 && y == eos)) {
      bad_token = true;
      continue;
    }
    consume_token(t, s, y, eos, max_len, root_has_children);
  }
  state[g] = s;
  if (bad_token && dev_status) atomicOr(dev_status, RGD_DEV_BAD_TOKEN);
  mask_rows(s, row_active, g, rows_per_group);
}

// ---------------------------------------------------------------------------
// Soft compatibility gate (the appendix ablation's Alg. 2), one probe step.
// In the first c steps, a greedy token y that would leave the refusal-prefix
// set does not end the probe at once: among the top-K tokens of the probe's
// next-token distribution (softmax of its logits; ties to the lower index),
// the refusal-compatible ones -- the children of the probe's trie node, and
// the stop token, which d(q) drops -- are found, and if their probability
// mass m reaches rho the most probable of them is appended instead.
//
// One block per group.  Pass 1 reads the probe's logits once: the maximum, its
// lowest index (y) and the softmax normaliser Z (per-thread online sums).  The
// soft branch then sorts the compatible candidates by logit in shared memory
// (bitonic sort of (logit, token) keys); their ranks grow along that order,
// so a binary search over it, one pass over the logits (from L2) per probed
// candidate, finds how many of them are in the top K.
constexpr int kSoftThreads = 512;
constexpr int kMaxCand = 2048;  // a node's children + the stop token, sorted in shared memory

struct SoftShared {
  uint64_t key[kMaxCand];
  float red_m[kSoftThreads / 32], red_z[kSoftThreads / 32];
  int32_t red_i[kSoftThreads / 32];
  int32_t cnt[1];
  rgd_gate_state s;
  float M, Z, mass;
  int32_t y, mode, ncand, n_in;
};

template <typename LT>
__device__ __forceinline__ float logit_at(const LT* row, int64_t i);
template <>
__device__ __forceinline__ float logit_at<float>(const float* row, int64_t i) {
  return __ldg(row + i);
}
template <>
__device__ __forceinline__ float logit_at<uint16_t>(const uint16_t* row, int64_t i) {
  return __uint_as_float((uint32_t)__ldg(row + i) << 16);
}

// Element e of a 16-byte vector of logits.
template <typename LT>
__device__ __forceinline__ float vec_elem(const uint4& w, int e);
template <>
__device__ __forceinline__ float vec_elem<float>(const uint4& w, int e) {
  return __uint_as_float(e == 0 ? w.x : e == 1 ? w.y : e == 2 ? w.z : w.w);
}
template <>
__device__ __forceinline__ float vec_elem<uint16_t>(const uint4& w, int e) {
  const uint32_t u = (e >> 1) == 0 ? w.x : (e >> 1) == 1 ? w.y : (e >> 1) == 2 ? w.z : w.w;
  return __uint_as_float((e & 1) ? (u & 0xffff0000u) : (u << 16));
}

// Calls f(logit, index) for this thread's share of a row, in increasing index
// order, with kBatchLoads loads in flight: 16-byte vectors when the row is
// 16-byte aligned (then the few elements past the last whole vector, one per
// thread, come last), else single elements.
template <int kThreads, int kBatchLoads, typename LT, typename F>
__device__ __forceinline__ void scan_row(const LT* row, int32_t vocab, bool vec, F&& f) {
  constexpr int E = 16 / (int)sizeof(LT);
  const int tid = threadIdx.x;
  if (vec) {
    const int32_t nvec = vocab / E;
    const uint4* rv = reinterpret_cast<const uint4*>(row);
    for (int32_t v0 = tid; v0 < nvec; v0 += kBatchLoads * kThreads) {
      uint4 w[kBatchLoads];
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b)
        if (v0 + b * kThreads < nvec) w[b] = __ldg(rv + v0 + b * kThreads);
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b) {
        const int32_t vi = v0 + b * kThreads;
        if (vi >= nvec) break;
#pragma unroll
        for (int e = 0; e < E; ++e) f(vec_elem<LT>(w[b], e), vi * E + e);
      }
    }
    const int32_t i = nvec * E + tid;
    if (i < vocab) f(logit_at<LT>(row, i), i);
  } else {
    for (int32_t i0 = tid; i0 < vocab; i0 += kBatchLoads * kThreads) {
      float v[kBatchLoads];
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b)
        if (i0 + b * kThreads < vocab) v[b] = logit_at<LT>(row, i0 + b * kThreads);
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b) {
        if (i0 + b * kThreads >= vocab) break;
        f(v[b], i0 + b * kThreads);
      }
    }
  }
}

// Order-preserving key: ascending keys = logits descending, then tokens ascending.
__device__ __forceinline__ uint64_t rank_key(float v, int32_t tok) {
  uint32_t u = __float_as_uint(v);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // ascending with v
  return ((uint64_t)(~u) << 32) | (uint32_t)tok;
}
__device__ __forceinline__ float key_logit(uint64_t k) {
  uint32_t u = ~(uint32_t)(k >> 32);
  u = (u & 0x80000000u) ? (u & 0x7fffffffu) : ~u;
  return __uint_as_float(u);
}

// (v, i) ranks above (w, j): a larger logit, or the same logit and a lower index.
__device__ __forceinline__ bool above(float v, int64_t i, float w, int64_t j) { return v > w || (v == w && i < j); }

template <typename LT>
__global__ void __launch_bounds__(kSoftThreads)
    soft_gate_kernel(TrieView t, int32_t rows_per_group, int32_t vocab, const LT* __restrict__ logits,
                     int64_t row_stride, bool vec, int32_t top_k, float rho, int32_t c, int32_t eos, int32_t max_len,
                     rgd_gate_state* __restrict__ state, uint8_t* __restrict__ row_active, int32_t* token_out,
                     float* mass_out) {
  __shared__ SoftShared sh;
  const int g = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const LT* row = logits + (int64_t)g * row_stride;
  if (tid == 0) {
    sh.s = state[g];
    sh.mode = 0;
    sh.mass = -1.f;
  }
  __syncthreads();
  if (sh.s.done) {  // (uniform) nothing to consume
    if (tid == 0) {
      token_out[g] = -1;
      if (mass_out) mass_out[g] = -1.f;
    }
    return;
  }
  // ---- pass 1: maximum, its lowest index, and Z = sum exp(l - max) ----
  float m = -INFINITY, z = 0.f;
  int32_t mi = 0x7fffffff;
  scan_row<kSoftThreads, 8, LT>(row, vocab, vec, [&](float v, int32_t i) {
    if (v > m) {  // indices grow along a thread: strict > keeps the lowest
      z = (m == -INFINITY) ? 1.f : z * expf(m - v) + 1.f;
      m = v;
      mi = i;
    } else if (m != -INFINITY) {  // (with m = -inf, v is -inf too and adds nothing)
      z += expf(v - m);
    }
  });
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m, o), oz = __shfl_xor_sync(0xffffffffu, z, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, mi, o);
    const float nm = fmaxf(m, om);
    z = (m == -INFINITY ? 0.f : z * expf(m - nm)) + (om == -INFINITY ? 0.f : oz * expf(om - nm));
    if (om > m || (om == m && oi < mi)) mi = oi;
    m = nm;
  }
  if (lane == 0) {
    sh.red_m[warp] = m;
    sh.red_z[warp] = z;
    sh.red_i[warp] = mi;
  }
  __syncthreads();
  if (tid == 0) {
    float M = sh.red_m[0], Z = sh.red_z[0];
    int32_t A = sh.red_i[0];
    for (int w = 1; w < kSoftThreads / 32; ++w) {
      const float om = sh.red_m[w], oz = sh.red_z[w];
      const float nm = fmaxf(M, om);
      Z = (M == -INFINITY ? 0.f : Z * expf(M - nm)) + (om == -INFINITY ? 0.f : oz * expf(om - nm));
      if (om > M || (om == M && sh.red_i[w] < A)) A = sh.red_i[w];
      M = nm;
    }
    sh.M = M;
    sh.Z = Z;
    sh.y = A;
    const rgd_gate_state& s = sh.s;
    const bool stop = eos >= 0 && A == eos;
    const bool compatible = s.confirmed || find_child(t, s.node, A) >= 0;
    sh.mode = (s.steps >= c || stop || compatible) ? 1 : 2;  // 1: the hard step with y; 2: the soft branch
    if (sh.mode == 2) {
      // the candidates: children of the node (and the stop token) inside the vocabulary
      const int32_t b = __ldg(t.child_begin + s.node), e = __ldg(t.child_begin + s.node + 1);
      int32_t n = 0;
      for (int32_t k = b; k < e; ++k) {
        const int32_t a = __ldg(t.child_tok + k);
        if (a >= 0 && a < vocab && a != eos) sh.key[n++] = rank_key(logit_at<LT>(row, a), a);
      }
      if (eos >= 0 && eos < vocab) sh.key[n++] = rank_key(logit_at<LT>(row, eos), eos);
      sh.ncand = n;
    }
  }
  __syncthreads();
  if (sh.mode == 2) {
    // ---- sort the candidates (bitonic, padded to a power of two) ----
    const int32_t n = sh.ncand;
    int32_t np = 1;
    while (np < n) np <<= 1;
    for (int32_t i = n + tid; i < np; i += kSoftThreads) sh.key[i] = ~0ull;
    __syncthreads();
    for (int32_t k = 2; k <= np; k <<= 1) {
      for (int32_t j = k >> 1; j > 0; j >>= 1) {
        for (int32_t i = tid; i < np; i += kSoftThreads) {
          const int32_t ij = i ^ j;
          if (ij > i) {
            const uint64_t a = sh.key[i], b2 = sh.key[ij];
            if ((a > b2) == ((i & k) == 0)) {
              sh.key[i] = b2;
              sh.key[ij] = a;
            }
          }
        }
        __syncthreads();
      }
    }
    // ---- how many of the sorted candidates are in the top K: their ranks
    // grow along the order, so a binary search, one candidate per pass (each
    // pass one comparison per logit, the logits read from L2) ----
    int32_t lo = 0, hi = min(n, top_k);
    while (lo < hi) {  // (lo, hi are the same in every thread)
      const int32_t mid = (lo + hi) >> 1;
      const uint64_t key = sh.key[mid];
      const float cv = key_logit(key);
      const int32_t ci = (int32_t)(uint32_t)key;
      if (tid == 0) sh.cnt[0] = 0;
      __syncthreads();
      int32_t cnt = 0;
      scan_row<kSoftThreads, 8, LT>(row, vocab, vec, [&](float v, int32_t i) { cnt += above(v, i, cv, ci) ? 1 : 0; });
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
      if (lane == 0 && cnt) atomicAdd(&sh.cnt[0], cnt);
      __syncthreads();
      if (sh.cnt[0] < top_k) lo = mid + 1;
      else hi = mid;
      __syncthreads();  // (sh.cnt is reset in the next pass)
    }
    if (tid == 0) {
      sh.n_in = lo;
      float mass = 0.f;
      for (int k = 0; k < lo; ++k) mass += expf(key_logit(sh.key[k]) - sh.M) / sh.Z;
      sh.mass = mass;
    }
    __syncthreads();
  }
  if (tid != 0) return;
  // ---- the step's outcome ----
  rgd_gate_state s = sh.s;
  const bool root_has_children = __ldg(t.child_begin + 1) > __ldg(t.child_begin);
  int32_t tok = -1;
  if (sh.mode == 1) {
    tok = sh.y;
    consume_token(t, s, tok, eos, max_len, root_has_children);
  } else if (sh.n_in > 0 && sh.mass >= rho) {
    tok = (int32_t)(uint32_t)sh.key[0];  // a*: the most probable compatible token
    consume_token(t, s, tok, eos, max_len, root_has_children);
  } else {  // no refusal-like alternative with enough mass: discard the probe
    s.decision = RGD_NON_REFUSAL;
    s.decisive_step = s.steps;
    s.steps++;
    s.done = 1;
  }
  state[g] = s;
  token_out[g] = tok;
  if (mass_out) mass_out[g] = sh.mode == 2 ? sh.mass : -1.f;
  mask_rows(s, row_active, g, rows_per_group);
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
  int32_t max_children = 0;
  for (int32_t n = 0; n < nn; ++n) {
    max_children = std::max(max_children, (int32_t)kids[n].size());
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
  t->max_children = max_children;
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

extern "C" int rgd_soft_gate(const rgd_trie* trie, int32_t groups, int32_t rows_per_group, int32_t vocab,
                             int32_t dtype, const void* probe_logits, int64_t row_stride, int32_t top_k, float rho,
                             int32_t c, int32_t eos_token, int32_t max_len, rgd_gate_state* state,
                             uint8_t* row_active, int32_t* token_out, float* mass_out, int32_t* dev_status,
                             rgd_stream_t stream) {
  clear_error();
  (void)dev_status;
  RGD_CHECK_ARG(trie != nullptr, "rgd_soft_gate: trie is NULL");
  RGD_CHECK_ARG(groups >= 0 && rows_per_group >= 1 && vocab >= 1, "rgd_soft_gate: bad groups/rows/vocab");
  RGD_CHECK_ARG(dtype == RGD_F32 || dtype == RGD_BF16, "rgd_soft_gate: dtype must be RGD_F32 or RGD_BF16");
  RGD_CHECK_ARG(row_stride >= vocab, "rgd_soft_gate: row_stride < vocab");
  RGD_CHECK_ARG(top_k >= 1 && c >= 0 && max_len >= 1, "rgd_soft_gate: need top_k >= 1, c >= 0, max_len >= 1");
  RGD_CHECK_ARG(std::isfinite(rho), "rgd_soft_gate: rho must be finite");
  if (trie->max_children + 1 > kMaxCand)
    return set_error(RGD_ERR_UNSUPPORTED, "rgd_soft_gate: a trie node has %d children (max %d)",
                     trie->max_children, kMaxCand - 1);
  if (groups == 0) return RGD_OK;
  RGD_CHECK_ARG(probe_logits != nullptr && state != nullptr && token_out != nullptr,
                "rgd_soft_gate: logits/state/token_out NULL");
  TrieView tv{trie->child_begin, trie->child_tok, trie->child_node, trie->confirm};
  cudaStream_t st = (cudaStream_t)stream;
  const int es = dtype == RGD_F32 ? 4 : 2;
  const bool vec = aligned16(probe_logits) && (row_stride * es) % 16 == 0;  // 16-byte vector loads
  if (dtype == RGD_F32)
    soft_gate_kernel<float><<<groups, kSoftThreads, 0, st>>>(tv, rows_per_group, vocab,
                                                              static_cast<const float*>(probe_logits), row_stride,
                                                              vec, top_k, rho, c, eos_token, max_len, state, row_active,
                                                              token_out, mass_out);
  else
    soft_gate_kernel<uint16_t><<<groups, kSoftThreads, 0, st>>>(tv, rows_per_group, vocab,
                                                                 static_cast<const uint16_t*>(probe_logits),
                                                                 row_stride, vec, top_k, rho, c, eos_token, max_len,
                                                                 state, row_active, token_out, mass_out);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "soft_gate launch");
}
