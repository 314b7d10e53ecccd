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
#include <cooperative_groups.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <map>
#include <mutex>
#include <vector>

#include "common.h"
#include "ptx.cuh"
#include "trie.cuh"

namespace rgd {
namespace cg = cooperative_groups;
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
// One thread-block cluster of kSoftCluster CTAs per group, each CTA taking an
// equal contiguous share of the probe's logits, copied into shared memory in
// chunks by bulk copies issued before anything else.  While they are in
// flight, the children of the probe's trie node (token, node, confirm flag)
// are read into shared memory -- every trie lookup of the step is then a
// shared-memory scan -- and, when the soft branch can be taken at this step,
// the candidates' keys (logit, token) and the kProbe best of them.  A
// candidate's rank -- the number of logits above it -- grows along the
// candidates' order, so the candidates in the top K are a prefix of that
// order.  The pass finds the maximum, its lowest index (y) and the softmax
// normaliser Z and counts the logits above each of the kProbe best
// candidates, which settles the prefix unless all of them are in the top K;
// then the candidates are sorted (bitonic, in shared memory) and a binary
// search over the rest, one more pass over the logits (from L2) per probed
// candidate, finishes it.  After each pass every CTA pushes its partial
// results into every CTA's shared memory and all of them combine the same
// values in the same order, so every CTA takes the same decisions; CTA 0
// writes the step's outcome.  The kernel runs once per decode step behind
// kernels that sweep L2, so its own instructions are fetched cold: its loops
// stay rolled, which keeps the code it runs short.
constexpr int kSoftThreads = 512;
constexpr int kSoftCluster = 6;
constexpr int kMaxCand = 2048;  // a node's children + the stop token (a power of two: the sort's padding)
constexpr int kProbe = 4;       // candidates whose ranks the first pass counts
constexpr int kSoftChunk = 32768;  // bytes of logits per bulk copy
constexpr int kSoftStages = 3;     // chunk buffers

struct SoftPart {  // one CTA's share of the first pass
  float m, z;
  int32_t mi;
  int32_t c[kProbe];
};

struct SoftShared {
  uint64_t key[kMaxCand];       // slot k < nc: child k; slot nc: the stop token (no candidate: ~0)
  int32_t slot_tok[kMaxCand];   // child k: its token, the node it leads to, that node's confirm flag
  int32_t slot_node[kMaxCand];
  uint8_t slot_conf[kMaxCand];
  SoftPart part[kSoftCluster * kSoftThreads / 32];  // first pass, slot = CTA rank x warps + warp
  int32_t cnt[2][kSoftCluster];  // search passes, slot = CTA rank, by pass parity
  int32_t cnt_cta;
  uint64_t full[kSoftStages];    // chunk buffer s holds its chunk
  int32_t ncand;
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

// Calls f(logit, index) for this thread's share of part `part` (of nparts
// equal contiguous parts) of a row, in increasing index order: 16-byte
// vectors when the row is 16-byte aligned (the few elements past the last
// whole vector, one per thread, go to the last part and come last), else
// single elements.  Every thread calls between() once, after its first batch
// of loads is issued and before any f (between() may hold block barriers).
template <int kThreads, int kBatchLoads, typename LT, typename F, typename B>
__device__ __forceinline__ void scan_row(const LT* row, int32_t vocab, bool vec, int part, int nparts, F&& f,
                                         B&& between) {
  constexpr int E = 16 / (int)sizeof(LT);
  const int tid = threadIdx.x;
  if (vec) {
    const int32_t nvec = vocab / E;
    const int32_t lo = (int32_t)((int64_t)nvec * part / nparts), hi = (int32_t)((int64_t)nvec * (part + 1) / nparts);
    const uint4* rv = reinterpret_cast<const uint4*>(row);
    uint4 w[kBatchLoads];
    int32_t v0 = lo + tid;
#pragma unroll
    for (int b = 0; b < kBatchLoads; ++b)
      if (v0 + b * kThreads < hi) w[b] = __ldg(rv + v0 + b * kThreads);
    between();
    for (;;) {
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b) {
        const int32_t vi = v0 + b * kThreads;
        if (vi >= hi) break;
#pragma unroll
        for (int e = 0; e < E; ++e) f(vec_elem<LT>(w[b], e), vi * E + e);
      }
      v0 += kBatchLoads * kThreads;
      if (v0 >= hi) break;
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b)
        if (v0 + b * kThreads < hi) w[b] = __ldg(rv + v0 + b * kThreads);
    }
    const int32_t i = nvec * E + tid;
    if (part == nparts - 1 && i < vocab) f(logit_at<LT>(row, i), i);
  } else {
    const int32_t lo = (int32_t)((int64_t)vocab * part / nparts), hi = (int32_t)((int64_t)vocab * (part + 1) / nparts);
    float v[kBatchLoads];
    int32_t i0 = lo + tid;
#pragma unroll
    for (int b = 0; b < kBatchLoads; ++b)
      if (i0 + b * kThreads < hi) v[b] = logit_at<LT>(row, i0 + b * kThreads);
    between();
    for (;;) {
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b) {
        if (i0 + b * kThreads >= hi) break;
        f(v[b], i0 + b * kThreads);
      }
      i0 += kBatchLoads * kThreads;
      if (i0 >= hi) break;
#pragma unroll
      for (int b = 0; b < kBatchLoads; ++b)
        if (i0 + b * kThreads < hi) v[b] = logit_at<LT>(row, i0 + b * kThreads);
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
__device__ __forceinline__ bool above(float v, int32_t i, float w, int32_t j) { return v > w || (v == w && i < j); }

constexpr float kLog2e = 1.4426950408889634f;

// Online softmax state (m, z, mi): the maximum logit seen, z = sum e^(l - m)
// over the logits seen (e^x = 2^(x log2 e), by the SFU), and the lowest index
// of the maximum.  Merges (om, oz, oi).
__device__ __forceinline__ void merge_mz(float& m, float& z, int32_t& mi, float om, float oz, int32_t oi) {
  const float nm = fmaxf(m, om);
  if (nm != -INFINITY) z = z * ex2_approx((m - nm) * kLog2e) + oz * ex2_approx((om - nm) * kLog2e);
  if (om > m || (om == m && oi < mi)) mi = oi;
  m = nm;
}

// The SoftParts of a warp's lanes, and n more from shared memory (n a multiple
// of 32: lane l folds parts[l], parts[l + 32], ...), merged in a fixed order;
// every lane returns lane 0's result.  One rolled loop, not inlined: every
// merge of the step runs the same few lines of code.
__device__ __noinline__ SoftPart merge_lanes(SoftPart p, const SoftPart* parts, int n) {
  const int lane = threadIdx.x & 31;
  int i = lane, o = 16;
#pragma unroll 1
  for (;;) {
    SoftPart q;
    if (i < n) {  // (uniform: n is a multiple of 32)
      q = parts[i];
      i += 32;
    } else if (o > 0) {
      q.m = __shfl_xor_sync(0xffffffffu, p.m, o);
      q.z = __shfl_xor_sync(0xffffffffu, p.z, o);
      q.mi = __shfl_xor_sync(0xffffffffu, p.mi, o);
#pragma unroll
      for (int k = 0; k < kProbe; ++k) q.c[k] = __shfl_xor_sync(0xffffffffu, p.c[k], o);
      o >>= 1;
    } else {
      break;
    }
    merge_mz(p.m, p.z, p.mi, q.m, q.z, q.mi);
#pragma unroll
    for (int k = 0; k < kProbe; ++k) p.c[k] += q.c[k];
  }
  p.m = __shfl_sync(0xffffffffu, p.m, 0);  // (the lanes may differ in z's rounding)
  p.z = __shfl_sync(0xffffffffu, p.z, 0);
  p.mi = __shfl_sync(0xffffffffu, p.mi, 0);
  return p;
}

template <typename LT>
__global__ void __cluster_dims__(kSoftCluster, 1, 1) __launch_bounds__(kSoftThreads, 1)
    soft_gate_kernel(TrieView t, int32_t rows_per_group, int32_t vocab, const LT* __restrict__ logits,
                     int64_t row_stride, bool vec, int32_t top_k, float rho, int32_t c, int32_t eos, int32_t max_len,
                     rgd_gate_state* __restrict__ state, uint8_t* __restrict__ row_active, int32_t* token_out,
                     float* mass_out, int32_t* dev_status) {
  constexpr int E = 16 / (int)sizeof(LT);   // logits per 16-byte vector
  constexpr int kVpc = kSoftChunk / 16;      // vectors per chunk
  constexpr int kWarps = kSoftThreads / 32;
  __shared__ SoftShared sh;
  extern __shared__ uint4 soft_buf[];  // kSoftStages chunks
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int g = blockIdx.x / kSoftCluster, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const LT* row = logits + (int64_t)g * row_stride;
  // this CTA's share of the row: vectors [lo, lo + nv) when the row is
  // 16-byte aligned (staged through shared memory), else elements [lo, hi_u)
  const int32_t nvec = vocab / E;
  const int32_t n_units = vec ? nvec : vocab;
  const int32_t lo = (int32_t)((int64_t)n_units * rank / kSoftCluster);
  const int32_t hi_u = (int32_t)((int64_t)n_units * (rank + 1) / kSoftCluster);
  const int32_t nv = vec ? hi_u - lo : 0;
  const int32_t nchunks = (nv + kVpc - 1) / kVpc;
  const uint4* rv = reinterpret_cast<const uint4*>(row);
  auto issue = [&](int32_t ck) {  // (thread 0) chunk ck into buffer ck % kSoftStages
    const uint32_t bytes = (uint32_t)min(kVpc, nv - ck * kVpc) * 16u;
    uint64_t* bar = &sh.full[ck % kSoftStages];
    mbar_arrive_expect_tx(bar, bytes);
    bulk_load(soft_buf + (ck % kSoftStages) * kVpc, rv + lo + ck * kVpc, bytes, bar);
  };
  bool timed_out = false;
  auto wait_chunk = [&](int32_t ck) {  // bounded; a second bounded wait after a timeout
    uint64_t* bar = &sh.full[ck % kSoftStages];
    const uint32_t par = (uint32_t)(ck / kSoftStages) & 1u;
    if (!mbar_wait(bar, par)) {
      timed_out = true;
      mbar_wait(bar, par);
    }
  };
  if (tid == 0) {
    for (int b = 0; b < kSoftStages; ++b) mbar_init(&sh.full[b], 1);
    fence_mbar_init();
    for (int32_t ck = 0; ck < min(kSoftStages, nchunks); ++ck) issue(ck);
    sh.ncand = 0;
  }
  // Every thread reads the state and takes the same decisions from it: the
  // kernel has no section where one warp works while the others wait.
  const rgd_gate_state s0 = state[g];
  __syncthreads();
  if (s0.done) {  // (uniform over the cluster) nothing to consume
    if (tid == 0) {
      for (int32_t ck = 0; ck < min(kSoftStages, nchunks); ++ck) wait_chunk(ck);  // (no copy outlives the CTA)
      if (timed_out && dev_status) atomicOr(dev_status, RGD_DEV_WAIT_TIMEOUT);
      if (rank == 0) {
        token_out[g] = -1;
        if (mass_out) mass_out[g] = -1.f;
      }
    }
    return;
  }
  cluster_arrive_relaxed();  // (waited for before the first push into another CTA)

  // ---- while the first chunks are in flight: the node's children (needed
  // unless the probe is confirmed) and, when the soft branch can be taken at
  // this step (the first c steps), the candidates' keys and the kProbe best ----
  const bool gather = !s0.confirmed;
  const bool maybe_soft = gather && s0.steps < c;
  int32_t cb = 0, nc = 0;
  if (gather) {
    cb = __ldg(t.child_begin + s0.node);
    nc = __ldg(t.child_begin + s0.node + 1) - cb;
  }
  const int32_t nslot = maybe_soft ? nc + 1 : nc;
  {
    int32_t mine = 0;
    for (int32_t k = tid; k < nslot; k += kSoftThreads) {
      int32_t a = eos;
      if (k < nc) {
        a = __ldg(t.child_tok + cb + k);
        const int32_t nd = __ldg(t.child_node + cb + k);
        sh.slot_tok[k] = a;
        sh.slot_node[k] = nd;
        sh.slot_conf[k] = __ldg(t.confirm + nd);
      }
      if (maybe_soft) {
        const bool ok = a >= 0 && a < vocab && (k == nc || a != eos);
        sh.key[k] = ok ? rank_key(logit_at<LT>(row, a), a) : ~0ull;
        mine += ok ? 1 : 0;
      }
    }
    if (mine) atomicAdd(&sh.ncand, mine);
  }
  __syncthreads();
  const int32_t n = sh.ncand;        // candidates
  const int32_t hi = min(n, top_k);  // only the first hi of them can be in the top K
  const int32_t np_ = min(hi, kProbe);
  // the np_ smallest keys (every warp finds them: one warp-wide minimum each;
  // keys are distinct); their logits and tokens probe the pass
  float pv[kProbe];
  int32_t pi[kProbe], pc[kProbe];
  {
    uint64_t prev = 0;
#pragma unroll
    for (int q = 0; q < kProbe; ++q) {
      uint64_t best = ~0ull;
      if (q < np_) {
#pragma unroll 1
        for (int32_t k = lane; k < nslot; k += 32) {
          const uint64_t key = sh.key[k];
          if ((q == 0 || key > prev) && key < best) best = key;
        }
        const uint32_t bh = __reduce_min_sync(0xffffffffu, (uint32_t)(best >> 32));
        const uint32_t bl = __reduce_min_sync(0xffffffffu, (uint32_t)(best >> 32) == bh ? (uint32_t)best : ~0u);
        best = ((uint64_t)bh << 32) | bl;
      }
      prev = best;
      pv[q] = q < np_ ? key_logit(best) : INFINITY;  // (nothing ranks above +inf at index 0)
      pi[q] = q < np_ ? (int32_t)(uint32_t)best : 0;
      pc[q] = 0;
    }
  }
  const float p_min = np_ > 0 ? pv[np_ - 1] : INFINITY;  // only a logit >= this can rank above a probe

  // ---- the pass: maximum, its lowest index, z = sum e^(l - m), probe ranks ----
  float m = -INFINITY, z = 0.f;
  int32_t mi = 0x7fffffff;
  auto probe_counts = [&](float v, int32_t i) {
#pragma unroll
    for (int q = 0; q < kProbe; ++q) pc[q] += above(v, i, pv[q], pi[q]) ? 1 : 0;
  };
  auto one = [&](float v, int32_t i) {  // a single logit (indices grow along a thread)
    if (v > m) {
      z = (m == -INFINITY) ? 0.f : z * ex2_approx((m - v) * kLog2e);
      m = v;
      mi = i;
    }
    if (m != -INFINITY) z += ex2_approx(fmaf(v, kLog2e, -m * kLog2e));
    if (v >= p_min) probe_counts(v, i);
  };
  if (vec) {
    for (int32_t ck = 0; ck < nchunks; ++ck) {
      wait_chunk(ck);
      const uint4* buf = soft_buf + (ck % kSoftStages) * kVpc;
      const int32_t cnt = min(kVpc, nv - ck * kVpc), base = lo + ck * kVpc;
      // this thread's vectors of the chunk: their maximum first, so that the
      // running maximum moves at most once per chunk
      float bm = -INFINITY;
#pragma unroll 1
      for (int32_t k = tid; k < cnt; k += kSoftThreads) {
        const uint4 x = buf[k];
#pragma unroll
        for (int e = 0; e < E; ++e) bm = fmaxf(bm, vec_elem<LT>(x, e));
      }
      if (bm > m) {  // the lowest index of bm here (indices grow along k, then e)
        int32_t bi = 0x7fffffff;
#pragma unroll 1
        for (int32_t k = tid; k < cnt && bi == 0x7fffffff; k += kSoftThreads) {
          const uint4 x = buf[k];
#pragma unroll
          for (int e = E - 1; e >= 0; --e)
            if (vec_elem<LT>(x, e) == bm) bi = (base + k) * E + e;
        }
        z = (m == -INFINITY) ? 0.f : z * ex2_approx((m - bm) * kLog2e);
        m = bm;
        mi = bi;
      }
      // z, and the probes for the few logits at or above the weakest one
      if (m != -INFINITY) {
        const float ml = m * kLog2e;
#pragma unroll 1
        for (int32_t k = tid; k < cnt; k += kSoftThreads) {
          const uint4 x = buf[k];
          float z0 = 0.f, z1 = 0.f;
#pragma unroll
          for (int e = 0; e < E; e += 2) {
            const float v0 = vec_elem<LT>(x, e), v1 = vec_elem<LT>(x, e + 1);
            z0 += ex2_approx(fmaf(v0, kLog2e, -ml));
            z1 += ex2_approx(fmaf(v1, kLog2e, -ml));
            if (v0 >= p_min) probe_counts(v0, (base + k) * E + e);
            if (v1 >= p_min) probe_counts(v1, (base + k) * E + e + 1);
          }
          z += z0 + z1;
        }
      } else if (bm >= p_min) {  // (every logit so far is -inf, and so is a probed candidate)
#pragma unroll 1
        for (int32_t k = tid; k < cnt; k += kSoftThreads) {
          const uint4 x = buf[k];
#pragma unroll
          for (int e = 0; e < E; ++e) probe_counts(vec_elem<LT>(x, e), (base + k) * E + e);
        }
      }
      if (ck + kSoftStages < nchunks) {
        __syncthreads();  // the buffer is free
        if (tid == 0) issue(ck + kSoftStages);
      }
    }
    // the few logits past the last whole vector
    const int32_t i = nvec * E + tid;
    if (rank == kSoftCluster - 1 && i < vocab) one(logit_at<LT>(row, i), i);
  } else {
    scan_row<kSoftThreads, 8, LT>(row, vocab, false, rank, kSoftCluster, one, [] {});
  }
  if (timed_out && dev_status) atomicOr(dev_status, RGD_DEV_WAIT_TIMEOUT);  // (the outputs are then not valid)

  // ---- every warp's share -> every CTA of the cluster ----
  {
    SoftPart p;
    p.m = m;
    p.z = z;
    p.mi = mi;
#pragma unroll
    for (int q = 0; q < kProbe; ++q) p.c[q] = pc[q];
    p = merge_lanes(p, nullptr, 0);
    cluster_wait();  // every CTA of the cluster has started
    if (lane < kSoftCluster) cluster.map_shared_rank(&sh, lane)->part[rank * kWarps + warp] = p;
  }
  cluster.sync();  // every warp's share is in every CTA's shared memory
  // ---- the same combination, in the same order, in every warp of the cluster ----
  SoftPart all;
  all.m = -INFINITY;
  all.z = 0.f;
  all.mi = 0x7fffffff;
#pragma unroll
  for (int q = 0; q < kProbe; ++q) all.c[q] = 0;
  all = merge_lanes(all, sh.part, kSoftCluster * kWarps);
  const int32_t y = all.mi;
  // the children labelled y and a* (the best candidate), if any
  const int32_t a_star = np_ > 0 ? pi[0] : -1;
  int32_t sy = -1, sa = -1;
#pragma unroll 1
  for (int32_t k = lane; k < nc; k += 32) {
    const int32_t tk = sh.slot_tok[k];
    if (tk == y) sy = k;  // (a node's children have distinct tokens)
    if (tk == a_star) sa = k;
  }
  sy = __reduce_max_sync(0xffffffffu, sy);
  sa = __reduce_max_sync(0xffffffffu, sa);
  const bool stop = eos >= 0 && y == eos;
  const bool compatible = s0.confirmed || sy >= 0;
  const bool soft = !(s0.steps >= c || stop || compatible);  // else the hard step with y
  // the probed candidates in the top K (a prefix: ranks grow along the order)
  int32_t n_in = 0;
  if (soft)
    while (n_in < np_ && all.c[n_in] < top_k) ++n_in;
  if (soft && n_in == np_ && np_ < hi) {
    // ---- the rest: sort the candidates (bitonic, padded to a power of two;
    // the first np_ are the probed ones), then a binary search over
    // candidates np_ .. hi - 1, one comparison per logit per probed
    // candidate (every thread of the cluster takes the same steps) ----
    int32_t np2 = 1;
    while (np2 < nslot) np2 <<= 1;
    for (int32_t i = nslot + tid; i < np2; i += kSoftThreads) sh.key[i] = ~0ull;
    __syncthreads();
    for (int32_t k = 2; k <= np2; k <<= 1) {
      for (int32_t j = k >> 1; j > 0; j >>= 1) {
        for (int32_t i = tid; i < np2; i += kSoftThreads) {
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
    int32_t lo_c = np_, hi_c = hi;
    for (int pass = 0; lo_c < hi_c; ++pass) {
      const int32_t mid = (lo_c + hi_c) >> 1;
      const uint64_t key = sh.key[mid];
      const float cv = key_logit(key);
      const int32_t ci = (int32_t)(uint32_t)key;
      if (tid == 0) sh.cnt_cta = 0;
      __syncthreads();
      int32_t cnt = 0;
      scan_row<kSoftThreads, 8, LT>(
          row, vocab, vec, rank, kSoftCluster, [&](float v, int32_t i) { cnt += above(v, i, cv, ci) ? 1 : 0; },
          [] {});
      cnt = __reduce_add_sync(0xffffffffu, cnt);
      if (lane == 0 && cnt) atomicAdd(&sh.cnt_cta, cnt);
      __syncthreads();
      // CTA r's slot of this pass's parity is next written two passes on,
      // after every CTA has passed the next cluster barrier (and read this one)
      if (warp == 0 && lane < kSoftCluster) cluster.map_shared_rank(&sh, lane)->cnt[pass & 1][rank] = sh.cnt_cta;
      cluster.sync();
      int32_t total = 0;
      for (int r = 0; r < kSoftCluster; ++r) total += sh.cnt[pass & 1][r];
      if (total < top_k) lo_c = mid + 1;
      else hi_c = mid;
    }
    n_in = lo_c;
  }
  // (no CTA touches another's shared memory after the last cluster barrier)
  if (warp != 0 || rank != 0) return;
  // ---- the step's outcome (warp 0 of CTA 0) ----
  float mass = -1.f;
  if (soft) {
    // m = the probability mass of the candidates in the top K
    const float ml = all.m * kLog2e;
    float part = 0.f;
    for (int32_t k = lane; k < n_in; k += 32) {
      float l = 0.f;
#pragma unroll
      for (int q = 0; q < kProbe; ++q)
        if (k == q) l = pv[q];
      if (k >= kProbe) l = key_logit(sh.key[k]);
      part += ex2_approx(fmaf(l, kLog2e, -ml));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    mass = part / all.z;
  }
  if (lane != 0) return;
  rgd_gate_state s = s0;
  auto child = [&](int32_t tok) {  // the gathered children: tok is y or a*
    const int32_t k = tok == y ? sy : sa;
    return k < 0 ? make_int2(-1, 0) : make_int2(sh.slot_node[k], (int)sh.slot_conf[k]);
  };
  const bool root_has_children = __ldg(t.child_begin + 1) > __ldg(t.child_begin);
  int32_t tok = -1;
  if (!soft) {
    tok = y;
    consume_token_with(s, tok, eos, max_len, root_has_children, child);
  } else if (n_in > 0 && mass >= rho) {
    tok = a_star;  // the most probable compatible token
    consume_token_with(s, tok, eos, max_len, root_has_children, child);
  } else {  // no refusal-like alternative with enough mass: discard the probe
    s.decision = RGD_NON_REFUSAL;
    s.decisive_step = s.steps;
    s.steps++;
    s.done = 1;
  }
  state[g] = s;
  token_out[g] = tok;
  if (mass_out) mass_out[g] = soft ? mass : -1.f;
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
  RGD_CHECK_ARG(trie != nullptr, "rgd_soft_gate: trie is NULL");
  RGD_CHECK_ARG(groups >= 0 && groups <= INT32_MAX / kSoftCluster && rows_per_group >= 1 && vocab >= 1,
                "rgd_soft_gate: bad groups/rows/vocab");
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
  constexpr int kDyn = kSoftStages * kSoftChunk;  // chunk buffers (dynamic shared memory)
  static std::once_flag attr_once;
  std::call_once(attr_once, [] {
    cudaFuncSetAttribute(soft_gate_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, kDyn);
    cudaFuncSetAttribute(soft_gate_kernel<uint16_t>, cudaFuncAttributeMaxDynamicSharedMemorySize, kDyn);
  });
  if (dtype == RGD_F32)
    soft_gate_kernel<float><<<groups * kSoftCluster, kSoftThreads, kDyn, st>>>(
        tv, rows_per_group, vocab, static_cast<const float*>(probe_logits), row_stride, vec, top_k, rho, c, eos_token,
        max_len, state, row_active, token_out, mass_out, dev_status);
  else
    soft_gate_kernel<uint16_t><<<groups * kSoftCluster, kSoftThreads, kDyn, st>>>(
        tv, rows_per_group, vocab, static_cast<const uint16_t*>(probe_logits), row_stride, vec, top_k, rho, c,
        eos_token, max_len, state, row_active, token_out, mass_out, dev_status);
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "soft_gate launch");
}
