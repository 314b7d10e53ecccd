// Shared-prefix split-KV decode attention.
//
// Sec. 3 reuses the prompt KV cache across the greedy probe and the high-
// temperature sampling stage.  Here that reuse is made explicit: the prompt KV
// of a group is read from HBM once per (kv head, split) and attended by all
// rows_per_group * (Hq/Hkv) queries of the group that map to that kv head; each
// row's own generated suffix is attended by that row's queries.  Partial results
// (unnormalised o, running max m, sum l) of every split are merged by
// log-sum-exp, which gives exactly attention over the concatenated KV.
//
// One CTA per work item (group|row, kv head, split):
//   * a producer warp streams the item's 16-token K/V page tiles into an
//     8-stage shared-memory ring with 2-D TMA loads (128-byte swizzle), paced by
//     full/empty mbarriers (all waits bounded);
//   * consumer warps each own 16 queries (one m16 tile) and a strided subset of
//     the pages; S = Q K^T and O += P V run on bf16 tensor-core MMAs with an
//     online softmax in fp32;
//   * the warps sharing a query tile are combined in shared memory and the
//     item's partial (o, m, l) goes to the workspace;
//   * the last item of a (group, kv head) to finish (atomic ticket, no waiting)
//     merges all partials of its queries, writes bf16 O and the fp32 LSE, and
//     resets the ticket.
#include <cudaTypedefs.h>

#include <cmath>
#include <mutex>

#include "common.h"
#include "ptx.cuh"

namespace rgd {
namespace {

constexpr int kPage = 16;
constexpr int kStages = 8;
constexpr int kConsumerWarps = 8;
constexpr int kAttnThreads = (kConsumerWarps + 1) * 32;
constexpr int kMaxQueries = 128;  // rows_per_group * Hq / Hkv per item
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct AttnParams {
  const __nv_bfloat16* q;
  const int32_t* prompt_bt;
  const int32_t* prompt_len;
  const int32_t* suffix_bt;
  const int32_t* suffix_len;
  const uint8_t* row_active;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;    // [R * Hq * NP, D]
  float2* part_ml;  // [R * Hq * NP]
  int32_t* ticket;  // [G * Hkv]
  int32_t* dev_status;
  int32_t G, rpg, Hq, Hkv, gq, num_pages;
  int32_t max_pp, max_sp;
  int32_t Sp, Ss, NP;
  int32_t n_prefix_items;
  float scale_log2;
};

template <int D>
struct Layout {
  static constexpr int kTileBytes = kPage * D * 2;               // one K (or V) page-head tile
  static constexpr int kStageBytes = 2 * kTileBytes;             // K + V
  static constexpr int kRingBytes = kStages * kStageBytes;
  static constexpr int kQStride = D * 2 + 16;                    // padded row (bank-conflict free)
  static constexpr int kQBytes = kMaxQueries * kQStride;
  static constexpr int kCombBytes = kConsumerWarps * 16 * (D + 2) * 4;
  static constexpr int kMainBytes = (kRingBytes + kQBytes) > kCombBytes ? (kRingBytes + kQBytes) : kCombBytes;
  static constexpr int kSmemBytes = kMainBytes + 1024 /* alignment slack */;
};

// Byte offset of (token t, 16-byte chunk c) in a page tile loaded as 64-column
// boxes with the 128-byte swizzle (chunk index XOR row index mod 8).
__device__ __forceinline__ uint32_t swz(uint32_t tile, int t, int c) {
  return tile + ((c >> 3) << 11) + (t << 7) + ((((c & 7) ^ (t & 7))) << 4);
}

__device__ __forceinline__ void flag(int32_t* status, int32_t bit) {
  if (status) atomicOr(status, bit);
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads, 2)
    attn_split_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                      const AttnParams p) {
  using L = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t full_bar[kStages], empty_bar[kStages];
  __shared__ int32_t s_flag_abort, s_issued, s_is_last;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  // ---- decode the work item ----------------------------------------------------
  const int item = blockIdx.x;
  const bool is_prefix = item < p.n_prefix_items;
  int g, h, s, row0, nq, part, S, n_tok, max_pages;
  const int32_t* bt;
  if (is_prefix) {
    s = item % p.Sp;
    h = (item / p.Sp) % p.Hkv;
    g = item / (p.Sp * p.Hkv);
    row0 = g * p.rpg;
    nq = p.rpg * p.gq;
    part = s;
    S = p.Sp;
    n_tok = p.prompt_len[g];
    max_pages = p.max_pp;
    bt = p.prompt_bt + (int64_t)g * p.max_pp;
  } else {
    const int it = item - p.n_prefix_items;
    s = it % p.Ss;
    h = (it / p.Ss) % p.Hkv;
    const int r = it / (p.Ss * p.Hkv);
    g = r / p.rpg;
    row0 = r;
    nq = p.gq;
    part = p.Sp + s;
    S = p.Ss;
    n_tok = p.suffix_len[r];
    max_pages = p.max_sp;
    bt = p.suffix_bt + (int64_t)r * p.max_sp;
  }
  if (n_tok < 0 || n_tok > max_pages * kPage) {
    if (tid == 0) flag(p.dev_status, RGD_DEV_BAD_PAGE);
    n_tok = n_tok < 0 ? 0 : max_pages * kPage;
  }
  // query i of this item -> (row, q head)
  auto q_row = [&](int i) { return is_prefix ? row0 + i / p.gq : row0; };
  auto q_head = [&](int i) { return h * p.gq + (is_prefix ? i % p.gq : i); };
  auto row_on = [&](int r) { return p.row_active == nullptr || p.row_active[r] != 0; };

  bool any_active = false;
  if (is_prefix) {
    for (int i = 0; i < p.rpg; ++i) any_active |= row_on(row0 + i);
  } else {
    any_active = row_on(row0);
  }
  const int n_pg_total = (n_tok + kPage - 1) / kPage;
  const int pps = (n_pg_total + S - 1) / S;
  const int page_begin = s * pps;
  const int n_pages = any_active ? max(0, min(n_pg_total, page_begin + pps) - page_begin) : 0;

  const int n_mt = (nq + 15) >> 4;
  const int TS = kConsumerWarps / n_mt;  // token slices (1, 2, 4 or 8)

  float* comb = reinterpret_cast<float*>(smem);  // [warp][16][D] then m,l, after the ring is drained
  float2* comb_ml = reinterpret_cast<float2*>(smem + kConsumerWarps * 16 * D * 4);
  const uint32_t ring = smem_u32(smem);
  uint8_t* qs = smem + L::kRingBytes;

  // per-consumer-warp online-softmax state (rows lane/4 and lane/4 + 8 of its tile)
  float o[D / 8][4];
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  const int col = 2 * (lane & 3);

  if (n_pages > 0) {
    if (tid == 0) {
      for (int i = 0; i < kStages; ++i) {
        mbar_init(&full_bar[i], 1);
        mbar_init(&empty_bar[i], n_mt);
      }
      s_flag_abort = 0;
      s_issued = 0;
      fence_mbar_init();
    }
    // queries of the item into shared memory; tile rows past nq are zero
    constexpr int kChunks = D / 8;
    for (int idx = tid; idx < n_mt * 16 * kChunks; idx += kAttnThreads) {
      const int i = idx / kChunks, c = idx % kChunks;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (i < nq)
        v = __ldg(reinterpret_cast<const uint4*>(p.q + ((int64_t)q_row(i) * p.Hq + q_head(i)) * D) + c);
      *reinterpret_cast<uint4*>(qs + i * L::kQStride + c * 16) = v;
    }
    __syncthreads();

    if (warp == kConsumerWarps) {
      // ---------------- producer ----------------
      if (lane == 0) {
        prefetch_tensormap(&tmK);
        prefetch_tensormap(&tmV);
        const uint64_t pol = policy_evict_first();
        int j = 0;
        for (; j < n_pages; ++j) {
          const int slot = j % kStages;
          if (j >= kStages && !mbar_wait(&empty_bar[slot], ((j / kStages) - 1) & 1)) {
            s_flag_abort = 1;
            break;
          }
          if (*(volatile int32_t*)&s_flag_abort) break;
          const int32_t page = __ldg(bt + page_begin + j);
          int32_t y = -2 * kPage;  // fully out of bounds: TMA fills zeros
          if (page >= 0 && page < p.num_pages) y = (page * p.Hkv + h) * kPage;
          else flag(p.dev_status, RGD_DEV_BAD_PAGE);
          uint8_t* kt = smem + slot * L::kStageBytes;
          mbar_arrive_expect_tx(&full_bar[slot], L::kStageBytes);
#pragma unroll
          for (int b = 0; b < D / 64; ++b) {
            tma_load_2d_hint(kt + b * 2048, &tmK, &full_bar[slot], b * 64, y, pol);
            tma_load_2d_hint(kt + L::kTileBytes + b * 2048, &tmV, &full_bar[slot], b * 64, y, pol);
          }
        }
        s_issued = j;
      }
    } else if (warp < n_mt * TS) {
      // ---------------- consumers ----------------
      const int mt = warp % n_mt, ts = warp / n_mt;
#pragma unroll
      for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
      const uint32_t qbase = smem_u32(qs) + (mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * L::kQStride +
                             (lane >> 4) * 16;
      const int kt_t = (lane & 7) + ((lane >> 4) & 1) * 8, kt_c = (lane >> 3) & 1;
      const int vt_t = (lane & 7) + ((lane >> 3) & 1) * 8, vt_c = lane >> 4;
      for (int j = ts; j < n_pages; j += TS) {
        const int slot = j % kStages;
        if (!mbar_wait(&full_bar[slot], (j / kStages) & 1)) {
          s_flag_abort = 1;
          break;
        }
        const uint32_t ktile = ring + slot * L::kStageBytes, vtile = ktile + L::kTileBytes;
        float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          uint32_t a[4], b[4];
          ldmatrix_x4(a, qbase + kk * 32);
          ldmatrix_x4(b, swz(ktile, kt_t, 2 * kk + kt_c));
          mma_bf16_16x8x16(sc[0], a, b[0], b[1]);
          mma_bf16_16x8x16(sc[1], a, b[2], b[3]);
        }
        const int valid = min(kPage, n_tok - (page_begin + j) * kPage);
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int t = nt * 8 + col + (e & 1);
            sc[nt][e] = (t < valid) ? sc[nt][e] * p.scale_log2 : -INFINITY;
          }
        float mx0 = fmaxf(fmaxf(sc[0][0], sc[0][1]), fmaxf(sc[1][0], sc[1][1]));
        float mx1 = fmaxf(fmaxf(sc[0][2], sc[0][3]), fmaxf(sc[1][2], sc[1][3]));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
        const float r0 = (n0 == -INFINITY) ? 0.f : n0, r1 = (n1 == -INFINITY) ? 0.f : n1;
        const float al0 = exp2f(m0 - r0), al1 = exp2f(m1 - r1);
        m0 = n0;
        m1 = n1;
        float pr[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
          pr[nt][0] = exp2f(sc[nt][0] - r0);
          pr[nt][1] = exp2f(sc[nt][1] - r0);
          pr[nt][2] = exp2f(sc[nt][2] - r1);
          pr[nt][3] = exp2f(sc[nt][3] - r1);
        }
        l0 = l0 * al0 + (pr[0][0] + pr[0][1] + pr[1][0] + pr[1][1]);
        l1 = l1 * al1 + (pr[0][2] + pr[0][3] + pr[1][2] + pr[1][3]);
#pragma unroll
        for (int i = 0; i < D / 8; ++i) {
          o[i][0] *= al0;
          o[i][1] *= al0;
          o[i][2] *= al1;
          o[i][3] *= al1;
        }
        uint32_t pa[4];
        pa[0] = pack_bf16x2(pr[0][0], pr[0][1]);
        pa[1] = pack_bf16x2(pr[0][2], pr[0][3]);
        pa[2] = pack_bf16x2(pr[1][0], pr[1][1]);
        pa[3] = pack_bf16x2(pr[1][2], pr[1][3]);
#pragma unroll
        for (int np = 0; np < D / 16; ++np) {
          uint32_t b[4];
          ldmatrix_x4_trans(b, swz(vtile, vt_t, 2 * np + vt_c));
          mma_bf16_16x8x16(o[2 * np], pa, b[0], b[1]);
          mma_bf16_16x8x16(o[2 * np + 1], pa, b[2], b[3]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[slot]);
      }
      l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
      l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
      l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    }
    // every copy has been consumed: the ring is reused for the combine buffers
    __syncthreads();
    if (warp < n_mt * TS && !s_flag_abort) {
      const int rr = lane >> 2;
      float* cw = comb + warp * 16 * D;
#pragma unroll
      for (int i = 0; i < D / 8; ++i) {
        const int d = i * 8 + col;
        cw[rr * D + d] = o[i][0];
        cw[rr * D + d + 1] = o[i][1];
        cw[(rr + 8) * D + d] = o[i][2];
        cw[(rr + 8) * D + d + 1] = o[i][3];
      }
      if ((lane & 3) == 0) {
        comb_ml[warp * 16 + rr] = make_float2(m0, l0);
        comb_ml[warp * 16 + rr + 8] = make_float2(m1, l1);
      }
    }
    __syncthreads();
    if (s_flag_abort) {
      // a copy did not land: wait (bounded) for the copies this block issued so
      // none is in flight at exit, report, and leave the outputs unwritten
      if (tid == 0) {
        flag(p.dev_status, RGD_DEV_WAIT_TIMEOUT);
        for (int j = max(0, s_issued - kStages); j < s_issued; ++j)
          mbar_wait(&full_bar[j % kStages], (j / kStages) & 1);
      }
      return;
    }
    // ---- combine the token slices of each query tile, write the item's partial --
    for (int idx = tid; idx < nq * D; idx += kAttnThreads) {
      const int i = idx / D, d = idx % D;
      if (!row_on(q_row(i))) continue;
      const int mt = i >> 4, rr = i & 15;
      float M = -INFINITY;
      for (int t = 0; t < TS; ++t) M = fmaxf(M, comb_ml[(t * n_mt + mt) * 16 + rr].x);
      float acc = 0.f, lsum = 0.f;
      if (M != -INFINITY) {
        for (int t = 0; t < TS; ++t) {
          const float2 ml = comb_ml[(t * n_mt + mt) * 16 + rr];
          const float w = exp2f(ml.x - M);
          acc += w * comb[((t * n_mt + mt) * 16 + rr) * D + d];
          lsum += w * ml.y;
        }
      }
      const int64_t pidx = ((int64_t)q_row(i) * p.Hq + q_head(i)) * p.NP + part;
      p.part_o[pidx * D + d] = acc;
      if (d == 0) p.part_ml[pidx] = make_float2(M, lsum);
    }
  } else {
    // empty or inactive item: an empty partial for every active query
    for (int i = tid; i < nq; i += kAttnThreads) {
      if (!row_on(q_row(i))) continue;
      const int64_t pidx = ((int64_t)q_row(i) * p.Hq + q_head(i)) * p.NP + part;
      p.part_ml[pidx] = make_float2(-INFINITY, 0.f);
    }
  }

  // ---- ticket: the last item of this (group, kv head) merges ------------------
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const int expected = p.Sp + p.rpg * p.Ss;
    const int prev = atomicAdd(p.ticket + g * p.Hkv + h, 1);
    s_is_last = (prev == expected - 1);
    if (s_is_last) __threadfence();
  }
  __syncthreads();
  if (!s_is_last) return;

  const int nwarps = kAttnThreads / 32;
  for (int qi = warp; qi < p.rpg * p.gq; qi += nwarps) {
    const int r = g * p.rpg + qi / p.gq, hq = h * p.gq + qi % p.gq;
    if (!row_on(r)) continue;
    const int64_t base = ((int64_t)r * p.Hq + hq) * p.NP;
    float M = -INFINITY;
    for (int i = 0; i < p.NP; ++i) M = fmaxf(M, __ldcg(&p.part_ml[base + i].x));
    constexpr int kPer = D / 32;
    float acc[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) acc[e] = 0.f;
    float lsum = 0.f;
    if (M != -INFINITY) {
      for (int i = 0; i < p.NP; ++i) {
        const float2 ml = __ldcg(&p.part_ml[base + i]);
        if (ml.y == 0.f) continue;
        const float w = exp2f(ml.x - M);
        lsum += w * ml.y;
        const float* po = p.part_o + (base + i) * D + lane * kPer;
        if constexpr (kPer == 4) {
          const float4 v = __ldcg(reinterpret_cast<const float4*>(po));
          acc[0] += w * v.x;
          acc[1] += w * v.y;
          acc[2] += w * v.z;
          acc[3] += w * v.w;
        } else {
          const float2 v = __ldcg(reinterpret_cast<const float2*>(po));
          acc[0] += w * v.x;
          acc[1] += w * v.y;
        }
      }
    }
    const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
    __nv_bfloat16* dst = p.out + (((int64_t)r * p.Hq + hq) * D) + lane * kPer;
    if constexpr (kPer == 4) {
      uint2 pk;
      pk.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
      pk.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(dst) = pk;
    } else {
      *reinterpret_cast<uint32_t*>(dst) = pack_bf16x2(acc[0] * inv, acc[1] * inv);
    }
    if (p.lse && lane == 0) p.lse[(int64_t)r * p.Hq + hq] = lsum > 0.f ? (M + log2f(lsum)) * kLn2 : -INFINITY;
  }
  __syncthreads();
  if (tid == 0) p.ticket[g * p.Hkv + h] = 0;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

int make_kv_map(CUtensorMap* map, const void* base, int64_t rows, int D) {
  auto fn = get_encode_fn();
  if (!fn) return set_error(RGD_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)D * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)kPage};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_error(RGD_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return RGD_OK;
}

struct Splits {
  int Sp, Ss;
};

Splits choose_splits(const rgd_attn_shape* s) {
  Splits sp;
  sp.Sp = s->prompt_splits > 0 ? s->prompt_splits : std::max(1, std::min(64, (s->max_prompt_pages + 31) / 32));
  sp.Ss = s->suffix_splits > 0 ? s->suffix_splits : std::max(1, std::min(64, (s->max_suffix_pages + 31) / 32));
  return sp;
}

struct WsLayout {
  size_t ticket_off, ml_off, o_off, total;
};

WsLayout ws_layout(const rgd_attn_shape* s) {
  const Splits sp = choose_splits(s);
  const int64_t R = (int64_t)s->num_groups * s->rows_per_group;
  const int64_t NP = sp.Sp + sp.Ss;
  const int64_t nparts = R * s->num_q_heads * NP;
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  WsLayout w;
  w.ticket_off = 0;
  w.ml_off = up((size_t)s->num_groups * s->num_kv_heads * sizeof(int32_t));
  w.o_off = w.ml_off + up((size_t)nparts * sizeof(float2));
  w.total = w.o_off + up((size_t)nparts * s->head_dim * sizeof(float));
  return w;
}

int check_shape(const rgd_attn_shape* s) {
  RGD_CHECK_ARG(s != nullptr, "attention shape is NULL");
  RGD_CHECK_ARG(s->num_groups >= 1 && s->rows_per_group >= 1, "num_groups and rows_per_group must be >= 1");
  RGD_CHECK_ARG(s->num_kv_heads >= 1 && s->num_q_heads >= s->num_kv_heads &&
                    s->num_q_heads % s->num_kv_heads == 0,
                "num_q_heads must be a positive multiple of num_kv_heads");
  if (s->head_dim != 64 && s->head_dim != 128)
    return set_error(RGD_ERR_UNSUPPORTED, "head_dim %d unsupported (64 or 128)", s->head_dim);
  if (s->page_size != kPage) return set_error(RGD_ERR_UNSUPPORTED, "page_size %d unsupported (16)", s->page_size);
  RGD_CHECK_ARG(s->num_pages >= 1, "num_pages must be >= 1");
  RGD_CHECK_ARG((int64_t)s->num_pages * s->num_kv_heads * kPage < (int64_t)1 << 31,
                "num_pages * num_kv_heads * page_size must be < 2^31");
  RGD_CHECK_ARG(s->max_prompt_pages >= 1 && s->max_suffix_pages >= 1, "block tables need >= 1 column");
  RGD_CHECK_ARG(s->prompt_splits >= 0 && s->suffix_splits >= 0, "split counts must be >= 0");
  const int nq = s->rows_per_group * (s->num_q_heads / s->num_kv_heads);
  if (nq > kMaxQueries)
    return set_error(RGD_ERR_UNSUPPORTED, "rows_per_group * Hq/Hkv = %d exceeds %d", nq, kMaxQueries);
  return RGD_OK;
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" size_t rgd_prefix_decode_attn_workspace_size(const rgd_attn_shape* shape) {
  clear_error();
  if (check_shape(shape) != RGD_OK) return 0;
  return ws_layout(shape).total;
}

extern "C" int rgd_prefix_decode_attn(const rgd_attn_shape* shape, const rgd_bf16* q, const rgd_bf16* k_pages,
                                      const rgd_bf16* v_pages, const int32_t* prompt_block_table,
                                      const int32_t* prompt_len, const int32_t* suffix_block_table,
                                      const int32_t* suffix_len, const uint8_t* row_active, float softmax_scale,
                                      rgd_bf16* out, float* lse, void* workspace, size_t workspace_bytes,
                                      int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  if (int rc = check_shape(shape)) return rc;
  const rgd_attn_shape& s = *shape;
  RGD_CHECK_ARG(q && k_pages && v_pages && prompt_block_table && prompt_len && suffix_block_table && suffix_len &&
                    out && workspace,
                "rgd_prefix_decode_attn: a required pointer is NULL");
  RGD_CHECK_ARG(aligned16(q) && aligned16(k_pages) && aligned16(v_pages) && aligned16(out),
                "rgd_prefix_decode_attn: q, k_pages, v_pages and out must be 16-byte aligned");
  RGD_CHECK_ARG((reinterpret_cast<uintptr_t>(workspace) & 255) == 0, "workspace must be 256-byte aligned");
  RGD_CHECK_ARG(std::isfinite(softmax_scale) && softmax_scale > 0.f, "softmax_scale must be > 0");
  const WsLayout w = ws_layout(shape);
  RGD_CHECK_ARG(workspace_bytes >= w.total, "workspace too small: %zu < %zu", workspace_bytes, w.total);
  const Splits sp = choose_splits(shape);

  CUtensorMap tmK, tmV;
  const int64_t kv_rows = (int64_t)s.num_pages * s.num_kv_heads * kPage;
  if (int rc = make_kv_map(&tmK, k_pages, kv_rows, s.head_dim)) return rc;
  if (int rc = make_kv_map(&tmV, v_pages, kv_rows, s.head_dim)) return rc;

  AttnParams p;
  p.q = reinterpret_cast<const __nv_bfloat16*>(q);
  p.prompt_bt = prompt_block_table;
  p.prompt_len = prompt_len;
  p.suffix_bt = suffix_block_table;
  p.suffix_len = suffix_len;
  p.row_active = row_active;
  p.out = reinterpret_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  p.ticket = reinterpret_cast<int32_t*>(ws + w.ticket_off);
  p.part_ml = reinterpret_cast<float2*>(ws + w.ml_off);
  p.part_o = reinterpret_cast<float*>(ws + w.o_off);
  p.dev_status = dev_status;
  p.G = s.num_groups;
  p.rpg = s.rows_per_group;
  p.Hq = s.num_q_heads;
  p.Hkv = s.num_kv_heads;
  p.gq = s.num_q_heads / s.num_kv_heads;
  p.num_pages = s.num_pages;
  p.max_pp = s.max_prompt_pages;
  p.max_sp = s.max_suffix_pages;
  p.Sp = sp.Sp;
  p.Ss = sp.Ss;
  p.NP = sp.Sp + sp.Ss;
  p.n_prefix_items = s.num_groups * s.num_kv_heads * sp.Sp;
  p.scale_log2 = softmax_scale * kLog2e;
  const int64_t R = (int64_t)s.num_groups * s.rows_per_group;
  const int64_t items = (int64_t)p.n_prefix_items + R * s.num_kv_heads * sp.Ss;
  RGD_CHECK_ARG(items < 0x7fffffff, "too many work items");

  cudaStream_t st = (cudaStream_t)stream;
  if (s.head_dim == 128) {
    static bool done = false;
    if (int rc = ensure_smem(attn_split_kernel<128>, Layout<128>::kSmemBytes, &done)) return rc;
    attn_split_kernel<128><<<(unsigned)items, kAttnThreads, Layout<128>::kSmemBytes, st>>>(tmK, tmV, p);
  } else {
    static bool done = false;
    if (int rc = ensure_smem(attn_split_kernel<64>, Layout<64>::kSmemBytes, &done)) return rc;
    attn_split_kernel<64><<<(unsigned)items, kAttnThreads, Layout<64>::kSmemBytes, st>>>(tmK, tmV, p);
  }
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "attention launch");
}

// ---------------------------------------------------------------------------
// Allocation-free variant of rgd_prefix_decode_attn
// ---------------------------------------------------------------------------
// The split partials and tickets live in a fixed file-scope device array
// instead of a caller-provided workspace.  The array exists once per device in
// every process that loads the library, for the life of the process.
namespace rgd {
namespace {

constexpr size_t kStaticScratchBytes = size_t(8) << 20;  // 8 MiB
__device__ __align__(256) uint8_t g_attn_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices] = {};

}  // namespace
}  // namespace rgd

extern "C" int rgd_prefix_decode_attn_noalloc(const rgd_attn_shape* shape, const rgd_bf16* q,
                                              const rgd_bf16* k_pages, const rgd_bf16* v_pages,
                                              const int32_t* prompt_block_table, const int32_t* prompt_len,
                                              const int32_t* suffix_block_table, const int32_t* suffix_len,
                                              const uint8_t* row_active, float softmax_scale, rgd_bf16* out,
                                              float* lse, int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  if (int rc = check_shape(shape)) return rc;
  const WsLayout w = ws_layout(shape);
  if (w.total > kStaticScratchBytes)
    return set_error(RGD_ERR_UNSUPPORTED,
                     "rgd_prefix_decode_attn_noalloc: this shape needs %zu bytes of scratch; the static "
                     "scratch holds %zu (use rgd_prefix_decode_attn with a workspace)",
                     w.total, kStaticScratchBytes);
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return set_error(RGD_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
  void* scratch = nullptr;
  {
    // once per device, with that device current: the host-side symbol is only a
    // stand-in, so the kernel gets the device address of the array
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_ptr[dev] == nullptr) {
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_attn_scratch);
      if (e != cudaSuccess) return cuda_error(e, "cudaGetSymbolAddress(g_attn_scratch)");
      g_scratch_ptr[dev] = p;
    }
    scratch = g_scratch_ptr[dev];
  }
  // the array keeps the previous call's contents: the tickets must start at zero
  e = cudaMemsetAsync(scratch, 0, w.ml_off, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_error(e, "cudaMemsetAsync(scratch tickets)");
  return rgd_prefix_decode_attn(shape, q, k_pages, v_pages, prompt_block_table, prompt_len, suffix_block_table,
                                suffix_len, row_active, softmax_scale, out, lse, scratch, kStaticScratchBytes,
                                dev_status, stream);
}
