// Sample head: the greedy step G_M and the truncated high-temperature sampler
// S_{T,theta} of Alg. 1, with min-p truncation and a Philox4x32-10 inverse-CDF
// draw.
//
// One thread-block cluster of kClusterCtas CTAs handles one row; the row is cut
// into equal contiguous ranges, one per warp of the cluster, and a warp reads
// its range as stripes of 32 coalesced 16-byte loads (kBatch stripes in flight
// per lane).  Pass 1 finds the row's max and lowest-index argmax (warp shuffles,
// shared memory, then distributed shared memory across the cluster).  Probe
// rows stop there.  Sample rows form the min-p cutoff from the max and, in
// pass 2, re-read their range (the row was read a moment ago and kept in L2) to
// sum the kept weights of every stripe (a lane's few elements in index order,
// then a butterfly across the lanes), keeping the stripe sums in shared memory.
// The Philox draw gives the target u * Z, and one warp walks the prefix sums in
// index order -- CTA, warp, stripe -- re-reads that single stripe and finds the
// lane and the element.  Sums are fp32 with compensation (a few ulp, well inside
// the 1e-6 of Z within which a draw counts as a boundary case); FP64 is slow on
// this part, so the only fp64 step is the cutoff's logarithm, once per row.
#include <cooperative_groups.h>

#include <cmath>

#include "common.h"
#include "ptx.cuh"
#include "trie.cuh"

namespace cg = cooperative_groups;

namespace rgd {
namespace {

constexpr int kClusterCtas = 8;
constexpr int kHeadThreads = 256;
constexpr int kHeadWarps = kHeadThreads / 32;
constexpr int kBatch = 4;        // 16-byte loads in flight per lane
constexpr int kMaxStripes = 64;  // stripes per warp whose sums are kept for the draw
constexpr int kSparseStripes = 16;  // stripes per warp for which lane maxima are kept
constexpr int kSparseHits = 16;     // vectors one lane re-reads at most in the sparse pass 2

struct HeadParams {
  const uint8_t* logits;
  int32_t rows;
  int32_t vocab;
  int32_t spw;  // stripes per warp
  const uint8_t* is_probe;
  const float* temperature;
  const float* min_p;
  const uint64_t* seed;
  uint64_t step;
  const uint8_t* row_active;
  int32_t* token_out;
  int32_t* kept_count;
  uint8_t* kept_mask;
  int32_t* dev_status;
  // the fused gate (gstate == nullptr: none): rows g * rpg .. g * rpg + rpg - 1
  // form group g, whose probe token (row g * rpg) goes through the hard gate
  TrieView trie;
  rgd_gate_state* gstate;
  uint8_t* gate_row_active;  // row_active, written by the gate
  int32_t rpg, eos, max_len;
};

// The fused gate.  The thread that writes a row's token then counts the row as
// finished in the top byte of its group's gate-state word {decision, confirmed,
// done, reserved}.  The probe row's thread first feeds its token to the hard
// gate (exactly rgd_probe_gate's step): it writes the state's integer fields
// directly and the decision, confirmed and done bytes by atomics, which leave
// the count in the top byte alone.  The group's last row to finish -- by then
// every row of the group has drawn its token and read its activity flag, and
// the probe's outcome is in the word its count returns -- masks the group's rows
// and sets the count back to zero.  Nothing waits, and the trie walk runs on
// the probe row, whose greedy path ends long before the sampled rows'.
__device__ __noinline__ void finish_row(const HeadParams& p, int row, int32_t tok) {
  const int g = row / p.rpg;
  rgd_gate_state* st = p.gstate + g;
  uint32_t* word = reinterpret_cast<uint32_t*>(&st->decision);
  if (row == g * p.rpg) {
    const uint32_t w0 = *reinterpret_cast<volatile uint32_t*>(word);  // (only this thread changes the low bytes)
    rgd_gate_state s;
    s.done = (uint8_t)((w0 >> 16) & 0xffu);
    if (!s.done) {
      if (tok < 0 && !(p.eos >= 0 && tok == p.eos)) {
        if (p.dev_status) atomicOr(p.dev_status, RGD_DEV_BAD_TOKEN);  // (an inactive or rejected probe row)
      } else {
        s.node = st->node;
        s.length = st->length;
        s.steps = st->steps;
        s.decisive_step = st->decisive_step;
        s.decision = (uint8_t)(w0 & 0xffu);
        s.confirmed = (uint8_t)((w0 >> 8) & 0xffu);
        const bool root_has_children = __ldg(p.trie.child_begin + 1) > __ldg(p.trie.child_begin);
        consume_token(p.trie, s, tok, p.eos, p.max_len, root_has_children);
        st->node = s.node;
        st->length = s.length;
        st->steps = s.steps;
        st->decisive_step = s.decisive_step;
        atomicAnd(word, 0xff000000u);
        atomicOr(word, (uint32_t)s.decision | ((uint32_t)s.confirmed << 8) | ((uint32_t)s.done << 16));
      }
    }
  }
  const uint32_t old = atomicAdd(word, 1u << 24);
  if ((int)(old >> 24) != p.rpg - 1) return;
  *word = old & 0x00ffffffu;  // the count back to 0 (every row of the group has counted itself)
  rgd_gate_state s;
  s.decision = (uint8_t)(old & 0xffu);
  s.done = (uint8_t)((old >> 16) & 0xffu);
  mask_rows(s, p.gate_row_active, g, p.rpg);
}

// 16 bytes of logits: 4 fp32 or 8 bf16 elements.
template <typename T>
struct Vec;
template <>
struct Vec<float> {
  static constexpr int kN = 4, kSize = 4;
  static constexpr uint32_t kNegInf = 0xff800000u, kNegInfWord = 0xff800000u;
  __device__ static float get(const uint4& w, int k) {
    const uint32_t u = k == 0 ? w.x : k == 1 ? w.y : k == 2 ? w.z : w.w;
    return __uint_as_float(u);
  }
  __device__ static uint32_t scalar(const uint8_t* p) { return *reinterpret_cast<const uint32_t*>(p); }
};
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int kN = 8, kSize = 2;
  static constexpr uint32_t kNegInf = 0xff80u, kNegInfWord = 0xff80ff80u;
  __device__ static float get(const uint4& w, int k) {
    const uint32_t u = (k >> 1) == 0 ? w.x : (k >> 1) == 1 ? w.y : (k >> 1) == 2 ? w.z : w.w;
    return __uint_as_float((k & 1) ? (u & 0xffff0000u) : (u << 16));
  }
  __device__ static uint32_t scalar(const uint8_t* p) { return *reinterpret_cast<const uint16_t*>(p); }
};

// The kN logits at element i of a row (i a multiple of kN); those at or past
// `vocab` read as -inf.  kAligned: the row starts 16-byte aligned and holds a
// whole number of 16-byte vectors.
template <typename T, bool kAligned>
__device__ __forceinline__ uint4 load_vec(const uint8_t* row, int64_t i, int32_t vocab, uint64_t policy) {
  using V = Vec<T>;
  if (kAligned) {
    if (i < vocab) return ld_nc_v4_hint(row + i * V::kSize, policy);
    return make_uint4(V::kNegInfWord, V::kNegInfWord, V::kNegInfWord, V::kNegInfWord);
  }
  uint32_t u[4];
  if (V::kSize == 4) {
#pragma unroll
    for (int k = 0; k < 4; ++k) u[k] = (i + k < vocab) ? V::scalar(row + (i + k) * 4) : V::kNegInf;
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint32_t lo = (i + 2 * k < vocab) ? V::scalar(row + (i + 2 * k) * 2) : V::kNegInf;
      const uint32_t hi = (i + 2 * k + 1 < vocab) ? V::scalar(row + (i + 2 * k + 1) * 2) : V::kNegInf;
      u[k] = lo | (hi << 16);
    }
  }
  return make_uint4(u[0], u[1], u[2], u[3]);
}

// Philox4x32-10 (Salmon et al., SC'11): word 0 of the block for (counter, key).
__device__ __forceinline__ uint32_t philox_word0(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                                 uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return c0;
}

// (value, index) order for the argmax: larger value wins, ties go to the lower index.
__device__ __forceinline__ bool better(float v, int32_t i, float bv, int32_t bi) {
  return v > bv || (v == bv && i < bi);
}

struct Shared {
  float red_v[kHeadWarps];
  int32_t red_i[kHeadWarps];
  float red_s[kHeadWarps];
  int32_t red_c[kHeadWarps];
  float stripe_sum[kHeadWarps][kMaxStripes];
  float stripe_max[kHeadWarps][kMaxStripes];
  // pass 1: each lane's maximum over its vector of each stripe (spw <=
  // kSparseStripes); pass 2 overwrites a lane's column with its partial sums
  float lane_part[kHeadWarps][kSparseStripes][33];
  uint8_t stripe_list[kHeadWarps][kMaxStripes];  // pass 2: the stripes a warp re-reads
  // pushed by every CTA of the cluster into every CTA's copy (slot = rank)
  float cta_max[kClusterCtas];
  int32_t cta_arg[kClusterCtas];
  float cta_sum[kClusterCtas];
  int32_t cta_cnt[kClusterCtas];
  // broadcast within the CTA
  float theta;  // T ln p_min (thread 0)
};

// Compensated (Kahan) fp32 running sum: the prefix sums of the draw stay within
// a few ulp of exact without fp64, which is slow on this part.
struct KSum {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float y = x - c;
    const float t = s + y;
    c = (t - s) - y;
    s = t;
  }
  __device__ __forceinline__ float value() const { return s - c; }
};

// The kept weight exp((l - M) / T) = 2^((l - M) log2(e) / T) of logit l, 0 below
// the cutoff; kexp = log2(e) / T per row.  The same fp32 steps everywhere, so
// pass 2 and the draw agree bit for bit.  Against exact weights the relative
// error is the factor's rounding times the exponent plus the 2^x unit's 2 ulp:
// a few 1e-7 for the weights that carry the mass (exponents near 0), inside the
// 1e-6 of Z within which a draw counts as a boundary case; weights below 2^-126
// flush to 0.
__device__ __forceinline__ float kept_weight(float l, float cut, float M, float kexp) {
  return l >= cut ? ex2_approx(__fsub_rn(l, M) * kexp) : 0.f;
}

template <typename T, bool kAligned>
__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kHeadThreads, 5)
    sample_head_kernel(const HeadParams p) {
  using V = Vec<T>;
  constexpr int kN = V::kN;
  constexpr int kStripe = 32 * kN;  // elements per stripe
  __shared__ Shared sh;
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int row = blockIdx.x / kClusterCtas;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // launched as a programmatic dependent of the previous kernel on the stream:
  // everything below may read what that kernel wrote
  asm volatile("griddepcontrol.wait;" ::: "memory");

  if (p.row_active && p.row_active[row] == 0) {  // uniform over the cluster
    if (rank == 0 && tid == 0) {
      p.token_out[row] = -1;
      if (p.kept_count) p.kept_count[row] = 0;
      if (p.gstate) finish_row(p, row, -1);
    }
    return;
  }
  cluster_arrive_relaxed();  // (waited for before the first push into another CTA)
  const uint8_t* rowp = p.logits + (int64_t)row * p.vocab * V::kSize;
  const int spw = p.spw;
  // warp w of CTA r reads stripes [(8r + w) spw, (8r + w + 1) spw) of the row
  auto elem = [&](int w, int s, int k) {
    return ((int64_t)(rank * kHeadWarps + w) * spw + s) * kStripe + lane * kN + k;
  };
  // the row is read again by pass 2 a few microseconds later: pass 1 asks L2 to
  // keep it, pass 2 (its last full read) lets it go
  const uint64_t keep_pol = policy_evict_last(), drop_pol = policy_evict_first();
  // the draw for this row, computed while the logits stream in
  // the row's parameters and the min-p offset T ln p_min (fp64 logarithm, one
  // thread) before pass 1, off the path after the row maximum
  const float temp = p.temperature[row];
  const float mp = p.min_p[row];
  const bool probe = p.is_probe && p.is_probe[row];
  float u = 0.f, theta = -INFINITY;
  if (tid == 0) {
    if (mp > 0.0f) theta = (float)((double)temp * log((double)mp));
    sh.theta = theta;  // (read after the first cluster barrier)
    const uint64_t sd = p.seed[row];
    const uint32_t x0 = philox_word0((uint32_t)p.step, (uint32_t)(p.step >> 32), 0u, 0u, (uint32_t)sd,
                                     (uint32_t)(sd >> 32));
    u = (float)(x0 >> 8) * (1.0f / 16777216.0f);  // exact: 24 bits
  }

  // ---- pass 1: max and lowest-index argmax ----------------------------------
  float bv = -INFINITY;
  int32_t bi = 0x7fffffff;
  for (int s0 = 0; s0 < spw; s0 += kBatch) {
    uint4 w[kBatch];
#pragma unroll
    for (int b = 0; b < kBatch; ++b)
      if (s0 + b < spw) w[b] = load_vec<T, kAligned>(rowp, elem(warp, s0 + b, 0), p.vocab, keep_pol);
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      if (s0 + b >= spw) break;
      const int32_t base = (int32_t)elem(warp, s0 + b, 0);
      float sm = -INFINITY;
#pragma unroll
      for (int k = 0; k < kN; ++k) {
        const float v = V::get(w[b], k);
        sm = fmaxf(sm, v);
        if (v > bv) {  // indices only grow along a lane: strict > keeps the lowest
          bv = v;
          bi = base + k;
        }
      }
      // the lane's and the stripe's maxima: pass 2 skips vectors and stripes
      // that cannot hold a kept token
      if (s0 + b < kSparseStripes) sh.lane_part[warp][s0 + b][lane] = sm;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sm = fmaxf(sm, __shfl_xor_sync(0xffffffffu, sm, o));
      if (lane == 0) sh.stripe_max[warp][s0 + b] = sm;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (better(ov, oi, bv, bi)) {
      bv = ov;
      bi = oi;
    }
  }
  if (lane == 0) {
    sh.red_v[warp] = bv;
    sh.red_i[warp] = bi;
  }
  cluster_wait();  // every CTA of the cluster has started
  __syncthreads();
  if (warp == 0) {
    float v = sh.red_v[0];
    int32_t i = sh.red_i[0];
    for (int w = 1; w < kHeadWarps; ++w)
      if (better(sh.red_v[w], sh.red_i[w], v, i)) {
        v = sh.red_v[w];
        i = sh.red_i[w];
      }
    // one lane per CTA of the cluster writes this CTA's maximum into that CTA
    if (lane < kClusterCtas) {
      Shared* o = cluster.map_shared_rank(&sh, lane);
      o->cta_max[rank] = v;
      o->cta_arg[rank] = i;
    }
  }
  // #1: every CTA's maximum is in every CTA's shared memory.  (All cluster
  // traffic is writes before a barrier and local reads after it, so no CTA
  // needs to outlive another's reads.)
  cluster.sync();
  // every warp merges the CTAs' maxima itself (no warp waits on another here)
  float M = -INFINITY;
  int32_t A = 0x7fffffff;
  if (lane < kClusterCtas) {
    M = sh.cta_max[lane];
    A = sh.cta_arg[lane];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, M, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, A, o);
    if (better(ov, oi, M, A)) {
      M = ov;
      A = oi;
    }
  }
  const bool greedy = probe || temp == 0.0f;
  const bool bad = !(temp >= 0.0f) || !isfinite(temp) || !(mp >= 0.0f && mp <= 1.0f) || !isfinite(M) ||
                   A >= p.vocab;
  if (greedy || bad) {
    if (rank == 0 && tid == 0) {
      int32_t tok = -1;
      if (bad && !greedy) {
        if (p.dev_status) atomicOr(p.dev_status, RGD_DEV_BAD_PARAM);
        if (p.kept_count) p.kept_count[row] = 0;
      } else {
        tok = A < p.vocab ? A : -1;
        if (p.kept_count) p.kept_count[row] = 1;
      }
      p.token_out[row] = tok;
      if (p.gstate) finish_row(p, row, tok);  // (this row is done: no further counting below)
    }
    return;
  }

  // ---- pass 2: kept weights; the sum of every stripe and of every warp -------
  const float cut = __fadd_rn(M, sh.theta);  // the min-p cutoff fl32(M + fl32(T ln p_min))
  const float kexp = 1.4426950408889634f / temp;
  uint8_t* mask = p.kept_mask ? p.kept_mask + (int64_t)row * p.vocab : nullptr;
  KSum wsum;  // identical in every lane
  int32_t cnt = 0;
  for (int st = lane; st < spw; st += 32) sh.stripe_sum[warp][st] = 0.f;
  // Sparse form: a lane's maxima from pass 1 say which of its vectors can hold
  // a kept token.  Every lane re-reads only its own such vectors (one trip to
  // L2 per four of them, instead of one per four stripes any lane hits), writes
  // each one's kept weight sum in its column of lane_part, and the warp sums
  // every stripe some lane hit.
  uint32_t hits = 0;
  bool sparse = mask == nullptr && spw <= kSparseStripes;
  if (sparse) {
    for (int st = 0; st < spw; ++st) hits |= sh.lane_part[warp][st][lane] >= cut ? (1u << st) : 0u;
    sparse = __all_sync(0xffffffffu, __popc(hits) <= kSparseHits);
  }
  if (sparse) {
    for (int st = 0; st < spw; ++st) sh.lane_part[warp][st][lane] = 0.f;
    uint32_t hm = hits;
    while (hm) {  // (lanes differ in their trip counts; no warp-wide operation inside)
      uint4 w[kBatch];
      int sidx[kBatch];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        sidx[b] = -1;
        if (hm) {
          sidx[b] = __ffs(hm) - 1;
          hm &= hm - 1;
          w[b] = load_vec<T, kAligned>(rowp, elem(warp, sidx[b], 0), p.vocab, drop_pol);
        }
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        if (sidx[b] < 0) break;
        const int32_t base = (int32_t)elem(warp, sidx[b], 0);
        uint32_t km = 0;
#pragma unroll
        for (int k = 0; k < kN; ++k) km |= (V::get(w[b], k) >= cut && base + k < p.vocab) ? (1u << k) : 0u;
        cnt += __popc(km);
        float ls = 0.f;
        while (km) {
          const int k = __ffs(km) - 1;
          km &= km - 1;
          ls += ex2_approx(__fsub_rn(V::get(w[b], k), M) * kexp);
        }
        sh.lane_part[warp][sidx[b]][lane] = ls;
      }
    }
    __syncwarp();
    // the sums of the stripes where some lane re-read a vector (the others stay 0),
    // each by a butterfly over the lanes (the same value in every lane), in stripe order
    uint32_t any = __reduce_or_sync(0xffffffffu, hits);
    while (any) {
      const int st = __ffs(any) - 1;
      any &= any - 1;
      float S = sh.lane_part[warp][st][lane];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
      if (lane == 0) sh.stripe_sum[warp][st] = S;
      wsum.add(S);
    }
  }
  // Dense form: only stripes whose maximum reaches the cutoff can hold a kept
  // token: the warp lists them (in index order) and re-reads just those; the
  // others' sums are 0.  With a kept mask requested every stripe is visited.
  int nlist = 0;
  for (int s0 = 0; s0 < spw && !sparse; s0 += 32) {
    const bool hit = s0 + lane < spw && (mask != nullptr || sh.stripe_max[warp][s0 + lane] >= cut);
    const uint32_t bal = __ballot_sync(0xffffffffu, hit);
    if (hit) sh.stripe_list[warp][nlist + __popc(bal & ((1u << lane) - 1u))] = (uint8_t)(s0 + lane);
    nlist += __popc(bal);
  }
  __syncwarp();
  for (int i0 = 0; i0 < nlist; i0 += kBatch) {
    uint4 w[kBatch];
    int sidx[kBatch];
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      sidx[b] = i0 + b < nlist ? sh.stripe_list[warp][i0 + b] : 0;
      if (i0 + b < nlist) w[b] = load_vec<T, kAligned>(rowp, elem(warp, sidx[b], 0), p.vocab, drop_pol);
    }
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      if (i0 + b >= nlist) break;
      const int32_t base = (int32_t)elem(warp, sidx[b], 0);
      // the lane's kept elements as a bit mask (the padding past the vocabulary reads -inf)
      uint32_t km = 0;
#pragma unroll
      for (int k = 0; k < kN; ++k) km |= (V::get(w[b], k) >= cut && base + k < p.vocab) ? (1u << k) : 0u;
      cnt += __popc(km);
      // weights in index order, one kept element per lane at a time: the warp
      // runs max-over-lanes rounds, not kN, and none where nothing is kept
      float ls = 0.f;
      while (km) {
        const int k = __ffs(km) - 1;
        km &= km - 1;
        ls += ex2_approx(__fsub_rn(V::get(w[b], k), M) * kexp);
      }
      if (mask) {
#pragma unroll
        for (int k = 0; k < kN; ++k)
          if (base + k < p.vocab) mask[base + k] = V::get(w[b], k) >= cut ? 1 : 0;
      }
      float S = ls;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
      if (lane == 0) sh.stripe_sum[warp][sidx[b]] = S;
      wsum.add(S);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if (lane == 0) {
    sh.red_s[warp] = wsum.value();
    sh.red_c[warp] = cnt;
  }
  __syncthreads();
  if (warp == 0) {
    KSum t;
    int32_t ct = 0;
    for (int w = 0; w < kHeadWarps; ++w) {
      t.add(sh.red_s[w]);
      ct += sh.red_c[w];
    }
    if (lane < kClusterCtas) {
      Shared* o = cluster.map_shared_rank(&sh, lane);
      o->cta_sum[rank] = t.value();
      o->cta_cnt[rank] = ct;
    }
  }
  cluster.sync();  // #2: every CTA's sums are in every CTA's shared memory
  // a sampled row other than the probe is counted by an idle warp, off the
  // draw's path (every CTA of the cluster read its activity flag long ago)
  if (p.gstate && rank == kClusterCtas - 1 && tid == 32 && row % p.rpg != 0) finish_row(p, row, -1);

  // ---- the draw: target u * Z; CTA, warp and stripe by prefix sums in index
  // order; then the stripe's lanes and the lane's elements --------------------
  float cs = 0.f;
  int32_t cc = 0;
  if (warp == 0 && lane < kClusterCtas) {
    cs = sh.cta_sum[lane];
    cc = sh.cta_cnt[lane];
  }
  if (warp == 0) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cc += __shfl_xor_sync(0xffffffffu, cc, o);
    // inclusive prefix sums in double over the lanes (a handful of values per row)
    auto scan = [&](double v) {
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const double t = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += t;
      }
      return v;
    };
    // the CTAs' sums in rank order: CTA r owns [incl(r-1), incl(r)), which tile [0, Z)
    const double ci = scan((double)cs);
    double ce = __shfl_up_sync(0xffffffffu, ci, 1);  // every lane takes part in the shuffle
    if (lane == 0) ce = 0.0;
    const double Z = __shfl_sync(0xffffffffu, ci, kClusterCtas - 1);
    const double target = (double)__shfl_sync(0xffffffffu, u, 0) * Z;
    const double lo = __shfl_sync(0xffffffffu, ce, rank), hi = __shfl_sync(0xffffffffu, ci, rank);
    const uint32_t nzc = __ballot_sync(0xffffffffu, lane < kClusterCtas && cs > 0.f);
    const float mine = __shfl_sync(0xffffffffu, cs, rank);
    if (lane == 0 && rank == 0 && p.kept_count) p.kept_count[row] = cc;
    if (mine > 0.f && lo <= target && (target < hi || rank == 31 - __clz(nzc))) {
      // the warp whose range holds the target (the last nonzero one if rounding
      // leaves the target past every range), then its stripe, the same way
      const float wsv = lane < kHeadWarps ? sh.red_s[lane] : 0.f;
      const double wi = lo + scan((double)wsv);
      const uint32_t whit = __ballot_sync(0xffffffffu, wsv > 0.f && target < wi);
      const uint32_t wnz = __ballot_sync(0xffffffffu, wsv > 0.f);
      int cw = whit ? __ffs(whit) - 1 : (wnz ? 31 - __clz(wnz) : 0);
      const double wbase = __shfl_sync(0xffffffffu, wi, cw) - (double)__shfl_sync(0xffffffffu, wsv, cw);
      int cst = -1, fb = -1;
      double sbase = wbase, run = wbase, fb_base = wbase;
      for (int s0 = 0; s0 < spw && cst < 0; s0 += 32) {
        const float sv = s0 + lane < spw ? sh.stripe_sum[cw][s0 + lane] : 0.f;
        const double si = run + scan((double)sv);
        const uint32_t shit = __ballot_sync(0xffffffffu, sv > 0.f && target < si);
        const uint32_t snz = __ballot_sync(0xffffffffu, sv > 0.f);
        const bool last = s0 + 32 >= spw;
        if (shit || (last && snz)) {
          const int L = shit ? __ffs(shit) - 1 : 31 - __clz(snz);
          cst = s0 + L;
          sbase = __shfl_sync(0xffffffffu, si, L) - (double)__shfl_sync(0xffffffffu, sv, L);
        } else if (snz) {
          // remember this round's last nonzero stripe in case rounding runs past the end
          const int L = 31 - __clz(snz);
          fb = s0 + L;
          fb_base = __shfl_sync(0xffffffffu, si, L) - (double)__shfl_sync(0xffffffffu, sv, L);
        }
        run = __shfl_sync(0xffffffffu, si, 31);
      }
      // (a warp or stripe is always found: a range with a nonzero sum has a
      // nonzero part; the guard only keeps a broken invariant from reading out of range)
      if (cst < 0 && fb >= 0) {
        cst = fb;
        sbase = fb_base;
      }
      if (cst < 0) cw = cst = 0;
      // the stripe's lanes: the same weights as pass 2, an inclusive scan in index order
      const uint4 w = load_vec<T, kAligned>(rowp, elem(cw, cst, 0), p.vocab, drop_pol);
      float ls = 0.f;
#pragma unroll
      for (int k = 0; k < kN; ++k) ls += kept_weight(V::get(w, k), cut, M, kexp);
      float incl = ls;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const uint32_t over = __ballot_sync(0xffffffffu, ls > 0.f && sbase + (double)incl > target);
      const uint32_t kept_lanes = __ballot_sync(0xffffffffu, ls > 0.f);
      const int L = over ? __ffs(over) - 1 : (kept_lanes ? 31 - __clz(kept_lanes) : 0);
      int32_t tok = -1;
      if (lane == L) {
        double r2 = sbase + (double)(incl - ls);
        int32_t lk = -1;
#pragma unroll
        for (int k = 0; k < kN; ++k) {
          const float wk = kept_weight(V::get(w, k), cut, M, kexp);
          if (wk > 0.f) {
            lk = (int32_t)elem(cw, cst, k);
            r2 += (double)wk;
            if (r2 > target && tok < 0) tok = lk;
          }
        }
        if (tok < 0) tok = lk;  // rounding put the target past the lane's last kept token
        if (tok < 0) tok = A;
        p.token_out[row] = tok;
        // (one lane of one CTA of the cluster writes the token; a sampled probe
        // row's token goes through the gate here)
        if (p.gstate && row % p.rpg == 0) finish_row(p, row, tok);
      }
    }
  }
}

}  // namespace
}  // namespace rgd

using namespace rgd;

namespace rgd {
namespace {

// The head kernel for the logits' type and alignment, launched as a
// programmatic dependent of the previous kernel on the stream, so that its
// blocks are scheduled while that kernel finishes (they wait for it before
// reading anything).
int launch_head(int32_t rows, int32_t vocab, int32_t dtype, const HeadParams& hp0, cudaStream_t st) {
  const int es = dtype == RGD_F32 ? 4 : 2;
  const int per_vec = 16 / es;
  const int64_t stripe = 32 * per_vec;
  const int64_t warps = (int64_t)kClusterCtas * kHeadWarps;
  HeadParams hp = hp0;
  hp.spw = (int32_t)((vocab + stripe * warps - 1) / (stripe * warps));
  const bool aligned = ((int64_t)vocab * es) % 16 == 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(rows * kClusterCtas);
  cfg.blockDim = dim3(kHeadThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e;
  if (dtype == RGD_F32)
    e = aligned ? cudaLaunchKernelEx(&cfg, sample_head_kernel<float, true>, hp)
                : cudaLaunchKernelEx(&cfg, sample_head_kernel<float, false>, hp);
  else
    e = aligned ? cudaLaunchKernelEx(&cfg, sample_head_kernel<__nv_bfloat16, true>, hp)
                : cudaLaunchKernelEx(&cfg, sample_head_kernel<__nv_bfloat16, false>, hp);
  if (e == cudaSuccess) e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "sample_head launch");
}

// Argument checks shared by both entry points.
int check_head_args(const char* fn, int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                    const float* temperature, const float* min_p, const uint64_t* seed, const int32_t* token_out) {
  RGD_CHECK_ARG(rows >= 0, "%s: rows < 0", fn);
  RGD_CHECK_ARG(vocab >= 1, "%s: vocab < 1", fn);
  RGD_CHECK_ARG(dtype == RGD_F32 || dtype == RGD_BF16, "%s: dtype must be RGD_F32 or RGD_BF16", fn);
  if (rows == 0) return RGD_OK;
  RGD_CHECK_ARG(logits && temperature && min_p && seed && token_out,
                "%s: logits/temperature/min_p/seed/token_out must be non-NULL", fn);
  RGD_CHECK_ARG(aligned16(logits), "%s: logits must be 16-byte aligned", fn);
  RGD_CHECK_ARG(rows <= 0x7fffffff / kClusterCtas, "%s: too many rows", fn);
  const int es = dtype == RGD_F32 ? 4 : 2;
  const int64_t stripe = 32 * (16 / es);
  const int64_t warps = (int64_t)kClusterCtas * kHeadWarps;
  if ((vocab + stripe * warps - 1) / (stripe * warps) > kMaxStripes)
    return set_error(RGD_ERR_UNSUPPORTED, "%s: vocab %d too large (max %lld)", fn, vocab,
                     (long long)(kMaxStripes * stripe * warps));
  return RGD_OK;
}

}  // namespace
}  // namespace rgd

extern "C" int rgd_sample_head(int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                               const uint8_t* is_probe, const float* temperature, const float* min_p,
                               const uint64_t* seed, uint64_t step, const uint8_t* row_active,
                               int32_t* token_out, int32_t* kept_count, uint8_t* kept_mask,
                               int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  if (int rc = check_head_args("rgd_sample_head", rows, vocab, dtype, logits, temperature, min_p, seed, token_out))
    return rc;
  if (rows == 0) return RGD_OK;
  HeadParams hp{static_cast<const uint8_t*>(logits), rows, vocab, 0, is_probe, temperature, min_p, seed,
                step, row_active, token_out, kept_count, kept_mask, dev_status};
  hp.gstate = nullptr;
  return launch_head(rows, vocab, dtype, hp, (cudaStream_t)stream);
}

namespace rgd {

int check_gated_head(const char* fn, int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                     const float* temperature, const float* min_p, const uint64_t* seed, const int32_t* token_out,
                     const rgd_trie* trie, int32_t rows_per_group, int32_t max_len, const rgd_gate_state* state) {
  if (int rc = check_head_args(fn, rows, vocab, dtype, logits, temperature, min_p, seed, token_out)) return rc;
  RGD_CHECK_ARG(trie != nullptr, "%s: trie is NULL", fn);
  RGD_CHECK_ARG(rows_per_group >= 1 && rows_per_group <= 255, "%s: rows_per_group must be in [1, 255]", fn);
  RGD_CHECK_ARG(rows % rows_per_group == 0, "%s: rows must be a multiple of rows_per_group", fn);
  RGD_CHECK_ARG(max_len >= 1, "%s: max_len must be >= 1", fn);
  if (rows == 0) return RGD_OK;
  RGD_CHECK_ARG(state != nullptr, "%s: state is NULL", fn);
  RGD_CHECK_ARG((reinterpret_cast<uintptr_t>(state) & 3u) == 0, "%s: state must be 4-byte aligned", fn);
  return RGD_OK;
}

}  // namespace rgd

extern "C" int rgd_sample_head_gated(int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                                     const uint8_t* is_probe, const float* temperature, const float* min_p,
                                     const uint64_t* seed, uint64_t step, uint8_t* row_active,
                                     int32_t* token_out, int32_t* kept_count, const rgd_trie* trie,
                                     int32_t rows_per_group, int32_t eos_token, int32_t max_len,
                                     rgd_gate_state* state, int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  if (int rc = check_gated_head("rgd_sample_head_gated", rows, vocab, dtype, logits, temperature, min_p, seed,
                                token_out, trie, rows_per_group, max_len, state))
    return rc;
  if (rows == 0) return RGD_OK;
  HeadParams hp{static_cast<const uint8_t*>(logits), rows, vocab, 0, is_probe, temperature, min_p, seed,
                step, row_active, token_out, kept_count, nullptr, dev_status};
  hp.trie = TrieView{trie->child_begin, trie->child_tok, trie->child_node, trie->confirm};
  hp.gstate = state;
  hp.gate_row_active = row_active;
  hp.rpg = rows_per_group;
  hp.eos = eos_token;
  hp.max_len = max_len;
  return launch_head(rows, vocab, dtype, hp, (cudaStream_t)stream);
}
