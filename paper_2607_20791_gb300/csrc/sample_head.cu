// Sample head: the greedy step G_M and the truncated high-temperature sampler
// S_{T,theta} of Alg. 1, with min-p truncation and a Philox4x32-10 inverse-CDF
// draw, reading every logit from HBM exactly once.
//
// One thread-block cluster of kClusterCtas CTAs handles one row.  Each CTA
// copies its contiguous slice of the row into shared memory with bulk copies
// (split into pieces so reduction starts while later pieces are in flight),
// reduces (max, lowest-index argmax) over its slice, and the CTAs exchange their
// results through distributed shared memory.  Sample rows then form the min-p
// cutoff from the row maximum, sum the kept weights of their slice from shared
// memory (no second HBM read), exchange the slice sums, and the one CTA whose
// cumulative range contains u * Z scans its slice for the drawn token.
#include <cooperative_groups.h>

#include <cmath>

#include "common.h"
#include "ptx.cuh"

namespace cg = cooperative_groups;

namespace rgd {
namespace {

constexpr int kClusterCtas = 8;
constexpr int kHeadThreads = 256;
constexpr int kHeadWarps = kHeadThreads / 32;
constexpr int kPieces = 4;
constexpr int kMaxSliceBytes = 200 * 1024;

struct HeadParams {
  const uint8_t* logits;
  int32_t rows;
  int32_t vocab;
  int32_t chunk;  // elements per CTA slice (multiple of 16)
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
};

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kSize = 4;
  __device__ static float load(const uint8_t* p) { return *reinterpret_cast<const float*>(p); }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kSize = 2;
  __device__ static float load(const uint8_t* p) {
    return __bfloat162float(*reinterpret_cast<const __nv_bfloat16*>(p));
  }
};

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
  uint64_t bar[kPieces];
  float red_v[kHeadWarps];
  int32_t red_i[kHeadWarps];
  double red_d[kHeadWarps];
  int32_t red_c[kHeadWarps];
  // published to the cluster
  float cta_max;
  int32_t cta_arg;
  double cta_sum;
  int32_t cta_cnt;
  // broadcast within the CTA
  float row_max;
  int32_t row_arg;
  double target;
  double cta_base;
  int32_t claim;
  int32_t bad;
};

template <typename T>
__global__ void __cluster_dims__(kClusterCtas, 1, 1) __launch_bounds__(kHeadThreads)
    sample_head_kernel(const HeadParams p) {
  using E = Elem<T>;
  constexpr int ES = E::kSize;
  __shared__ Shared sh;
  extern __shared__ __align__(128) uint8_t dyn[];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int row = blockIdx.x / kClusterCtas;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  if (p.row_active && p.row_active[row] == 0) {  // uniform over the cluster
    if (rank == 0 && tid == 0) {
      p.token_out[row] = -1;
      if (p.kept_count) p.kept_count[row] = 0;
    }
    return;
  }

  // ---- slice of the row owned by this CTA ---------------------------------
  const int32_t e0 = min(p.vocab, rank * p.chunk);
  const int32_t e1 = min(p.vocab, e0 + p.chunk);
  const int32_t n = e1 - e0;
  const uint8_t* gsrc = p.logits + ((int64_t)row * p.vocab + e0) * ES;
  const uint32_t mis = (uint32_t)(reinterpret_cast<uintptr_t>(gsrc) & 15u);
  const int32_t head_el = min(n, (int32_t)(((16u - mis) & 15u) / ES));
  const uint32_t int_bytes = (uint32_t)((n - head_el) * ES) & ~15u;
  const int32_t int_el = (int32_t)(int_bytes / ES);
  // sbuf[k] holds element e0 + k; the bulk-copied interior starts 16-byte aligned
  uint8_t* sbuf = dyn + ((16u - (uint32_t)(head_el * ES)) & 15u);
  const uint32_t piece = ((int_bytes + kPieces - 1) / kPieces + 15u) & ~15u;

  if (tid == 0) {
    for (int k = 0; k < kPieces; ++k) mbar_init(&sh.bar[k], 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {
    for (int k = 0; k < kPieces; ++k) {
      const uint32_t b = k * piece;
      if (b >= int_bytes) break;
      const uint32_t sz = min(piece, int_bytes - b);
      mbar_arrive_expect_tx(&sh.bar[k], sz);
      bulk_load(sbuf + head_el * ES + b, gsrc + head_el * ES + b, sz, &sh.bar[k]);
    }
  }

  // ---- phase 1: max and lowest-index argmax of the slice ---------------------
  float bv = -INFINITY;
  int32_t bi = 0x7fffffff;
  // ragged edges (fewer than 16 bytes each) with plain loads
  for (int32_t k = tid; k < n - int_el; k += kHeadThreads) {
    const int32_t idx = (k < head_el) ? k : (head_el + int_el + (k - head_el));
    const float v = E::load(gsrc + idx * ES);
    *reinterpret_cast<T*>(sbuf + idx * ES) = *reinterpret_cast<const T*>(gsrc + idx * ES);
    if (better(v, e0 + idx, bv, bi)) { bv = v; bi = e0 + idx; }
  }
  bool timed_out = false;
  for (int k = 0; k < kPieces; ++k) {
    const uint32_t b = k * piece;
    if (b >= int_bytes) break;
    const uint32_t sz = min(piece, int_bytes - b);
    // bounded: a copy that never lands is reported, and the later pieces are
    // still waited for (again bounded) so no copy is in flight at exit
    if (!mbar_wait(&sh.bar[k], 0)) {
      timed_out = true;
      continue;
    }
    if (timed_out) continue;
    const uint8_t* base = sbuf + head_el * ES + b;
    const int32_t el_base = head_el + (int32_t)(b / ES);
    for (uint32_t off = tid * 16u; off < sz; off += kHeadThreads * 16u) {
      const uint4 w = *reinterpret_cast<const uint4*>(base + off);
      const int32_t i0 = e0 + el_base + (int32_t)(off / ES);
      if constexpr (ES == 4) {
        const float v[4] = {__uint_as_float(w.x), __uint_as_float(w.y), __uint_as_float(w.z),
                            __uint_as_float(w.w)};
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (better(v[j], i0 + j, bv, bi)) { bv = v[j]; bi = i0 + j; }
      } else {
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float lo = __uint_as_float(u[j] << 16), hi = __uint_as_float(u[j] & 0xffff0000u);
          if (better(lo, i0 + 2 * j, bv, bi)) { bv = lo; bi = i0 + 2 * j; }
          if (better(hi, i0 + 2 * j + 1, bv, bi)) { bv = hi; bi = i0 + 2 * j + 1; }
        }
      }
    }
  }
  // the row's outputs are invalid after a timeout; the protocol still runs to
  // its end so that every CTA of the cluster meets the same cluster barriers
  if (timed_out && tid == 0 && p.dev_status) atomicOr(p.dev_status, RGD_DEV_WAIT_TIMEOUT);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int32_t oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
  }
  if (lane == 0) {
    sh.red_v[warp] = bv;
    sh.red_i[warp] = bi;
  }
  __syncthreads();
  if (tid == 0) {
    float v = sh.red_v[0];
    int32_t i = sh.red_i[0];
    for (int w = 1; w < kHeadWarps; ++w)
      if (better(sh.red_v[w], sh.red_i[w], v, i)) { v = sh.red_v[w]; i = sh.red_i[w]; }
    sh.cta_max = v;
    sh.cta_arg = i;
  }
  cluster.sync();  // #1: slice maxima visible to the cluster
  if (tid == 0) {
    float v = -INFINITY;
    int32_t i = 0x7fffffff;
    for (int r = 0; r < kClusterCtas; ++r) {
      const Shared* o = cluster.map_shared_rank(&sh, r);
      if (better(o->cta_max, o->cta_arg, v, i)) { v = o->cta_max; i = o->cta_arg; }
    }
    sh.row_max = v;
    sh.row_arg = i;
  }
  __syncthreads();
  const float M = sh.row_max;
  const int32_t A = sh.row_arg;
  const float temp = p.temperature[row];
  const float mp = p.min_p[row];
  const bool greedy = (p.is_probe && p.is_probe[row]) || temp == 0.0f;
  const bool bad = !(temp >= 0.0f) || !isfinite(temp) || !(mp >= 0.0f && mp <= 1.0f) || !isfinite(M) ||
                   A >= p.vocab;
  if (greedy || bad) {
    if (rank == 0 && tid == 0) {
      if (bad && !greedy) {
        if (p.dev_status) atomicOr(p.dev_status, RGD_DEV_BAD_PARAM);
        p.token_out[row] = -1;
        if (p.kept_count) p.kept_count[row] = 0;
      } else {
        p.token_out[row] = A < p.vocab ? A : -1;
        if (p.kept_count) p.kept_count[row] = 1;
      }
    }
    cluster.sync();  // keep this CTA's shared memory alive until every CTA has read it
    return;
  }

  // ---- phase 2: min-p cutoff and kept weights of this CTA's slice -------------
  const float theta = (mp > 0.0f) ? (float)((double)temp * log((double)mp)) : -INFINITY;
  const float cut = __fadd_rn(M, theta);
  const int32_t per = (n + kHeadThreads - 1) / kHeadThreads;
  const int32_t k0 = min(n, tid * per), k1 = min(n, k0 + per);
  float s = 0.0f, comp = 0.0f;  // Kahan-compensated sum of this thread's kept weights
  int32_t cnt = 0;
  uint8_t* mask = p.kept_mask ? p.kept_mask + (int64_t)row * p.vocab + e0 : nullptr;
  for (int32_t k = k0; k < k1; ++k) {
    const float l = E::load(sbuf + k * ES);
    const bool keep = l >= cut;
    if (mask) mask[k] = keep ? 1 : 0;
    if (keep) {
      const float w = expf(__fdiv_rn(__fsub_rn(l, M), temp));
      const float y = w - comp;
      const float t2 = s + y;
      comp = (t2 - s) - y;
      s = t2;
      ++cnt;
    }
  }
  // exclusive scan of the per-thread sums (double) across the CTA
  // inclusive warp scan; the exclusive prefix is the previous lane's inclusive
  // value, so consecutive thread boundaries are monotone and partition exactly
  double incl = (double)s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  double prev = __shfl_up_sync(0xffffffffu, incl, 1);
  if (lane == 0) prev = 0.0;
  int32_t c = cnt;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  if (lane == 31) sh.red_d[warp] = incl;
  if (lane == 0) sh.red_c[warp] = c;
  __syncthreads();
  double warp_base = 0.0;
  for (int w = 0; w < warp; ++w) warp_base += sh.red_d[w];
  const double excl = warp_base + prev;
  if (tid == 0) {
    double tot = 0.0;
    int32_t ct = 0;
    for (int w = 0; w < kHeadWarps; ++w) {
      tot += sh.red_d[w];
      ct += sh.red_c[w];
    }
    sh.cta_sum = tot;
    sh.cta_cnt = ct;
  }
  cluster.sync();  // #2: slice sums visible to the cluster
  if (tid == 0) {
    double base = 0.0, mine = 0.0;
    int32_t count = 0;
    for (int r = 0; r < kClusterCtas; ++r) {
      const Shared* o = cluster.map_shared_rank(&sh, r);
      if (r == rank) mine = base;
      base += o->cta_sum;
      count += o->cta_cnt;
    }
    const uint64_t sd = p.seed[row];
    const uint32_t x0 = philox_word0((uint32_t)p.step, (uint32_t)(p.step >> 32), 0u, 0u, (uint32_t)sd,
                                     (uint32_t)(sd >> 32));
    const double u = (double)(x0 >> 8) * (1.0 / 16777216.0);
    const double target = u * base;
    sh.target = target;
    sh.cta_base = mine;
    sh.claim = (mine <= target && target < mine + sh.cta_sum) ? 1 : 0;
    if (rank == 0 && p.kept_count) p.kept_count[row] = count;
  }
  __syncthreads();
  if (sh.claim) {
    const double target = sh.target;
    const double lo = sh.cta_base + excl;
    // the next thread's boundary; the last thread's is the CTA's upper end
    double hi = __shfl_down_sync(0xffffffffu, lo, 1);
    if (lane == 31) hi = (warp + 1 < kHeadWarps) ? sh.cta_base + (warp_base + sh.red_d[warp])
                                                   : sh.cta_base + sh.cta_sum;
    if (lo <= target && target < hi) {
      double run = lo;
      int32_t tok = -1, last = -1;
      for (int32_t k = k0; k < k1; ++k) {
        const float l = E::load(sbuf + k * ES);
        if (l >= cut) {
          last = k;
          run += (double)expf(__fdiv_rn(__fsub_rn(l, M), temp));
          if (run > target) {
            tok = k;
            break;
          }
        }
      }
      if (tok < 0) tok = last;
      p.token_out[row] = e0 + tok;
    }
  }
  cluster.sync();  // #3: shared memory stays alive until the cluster is done reading it
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" int rgd_sample_head(int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                               const uint8_t* is_probe, const float* temperature, const float* min_p,
                               const uint64_t* seed, uint64_t step, const uint8_t* row_active,
                               int32_t* token_out, int32_t* kept_count, uint8_t* kept_mask,
                               int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  RGD_CHECK_ARG(rows >= 0, "rgd_sample_head: rows < 0");
  RGD_CHECK_ARG(vocab >= 1, "rgd_sample_head: vocab < 1");
  RGD_CHECK_ARG(dtype == RGD_F32 || dtype == RGD_BF16, "rgd_sample_head: dtype must be RGD_F32 or RGD_BF16");
  if (rows == 0) return RGD_OK;
  RGD_CHECK_ARG(logits && temperature && min_p && seed && token_out,
                "rgd_sample_head: logits/temperature/min_p/seed/token_out must be non-NULL");
  RGD_CHECK_ARG(aligned16(logits), "rgd_sample_head: logits must be 16-byte aligned");
  RGD_CHECK_ARG(rows <= 0x7fffffff / kClusterCtas, "rgd_sample_head: too many rows");
  const int es = dtype == RGD_F32 ? 4 : 2;
  const int32_t chunk = ((vocab + kClusterCtas - 1) / kClusterCtas + 15) & ~15;
  const int smem = chunk * es + 32;
  if (chunk * es > kMaxSliceBytes)
    return set_error(RGD_ERR_UNSUPPORTED, "rgd_sample_head: vocab %d too large (max slice %d bytes)", vocab,
                     kMaxSliceBytes);
  HeadParams hp{static_cast<const uint8_t*>(logits), rows, vocab, chunk, is_probe, temperature, min_p, seed,
                step, row_active, token_out, kept_count, kept_mask, dev_status};
  const dim3 grid(rows * kClusterCtas), block(kHeadThreads);
  cudaStream_t st = (cudaStream_t)stream;
  if (dtype == RGD_F32) {
    static bool done = false;
    if (int rc = ensure_smem(sample_head_kernel<float>, kMaxSliceBytes + 32, &done)) return rc;
    sample_head_kernel<float><<<grid, block, smem, st>>>(hp);
  } else {
    static bool done = false;
    if (int rc = ensure_smem(sample_head_kernel<__nv_bfloat16>, kMaxSliceBytes + 32, &done)) return rc;
    sample_head_kernel<__nv_bfloat16><<<grid, block, smem, st>>>(hp);
  }
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "sample_head launch");
}
