// Shared-prefix decode attention: persistent, balanced, one pass over the KV.
//
// Sec. 3 reuses the prompt KV cache across the greedy probe and the high-
// temperature sampling stage.  Here that reuse is explicit: for every prompt
// group g and kv head h one "job" attends all rows_per_group * (Hq/Hkv) queries
// of the group that map to h.  A job's page list is the group's prompt pages
// (visible to every row) followed by the suffix pages of each active row
// (visible to that row's queries only, by a per-page row mask), so a row's
// suffix simply continues the online softmax of its prompt: the result is
// attention over [prompt KV | own suffix KV], and every KV page is read from
// HBM exactly once.
//
// Work distribution.  The jobs' page lists are laid end to end (job-major) and
// the grid's persistent CTAs (one per SM) each take an equal contiguous range of
// pages.  Inside a CTA a producer warp streams its pages' 16-token K/V tiles into
// a shared-memory ring with 2-D TMA loads (128-byte swizzle), across job
// boundaries, paced by full/empty mbarriers whose waits are all bounded.  Fifteen
// consumer warps own (query tile of 16, token slice) pairs and run S = Q K^T and
// O += P V on bf16 tensor-core MMAs with an online softmax in fp32.  At the end
// of each job piece the token slices are combined in shared memory; a job that
// lies inside one CTA is written out directly, a job split across CTAs leaves a
// partial (o, m, l) in workspace slot (cta + job) -- distinct for every piece,
// since CTA ranges are ordered like the jobs -- and the last piece to finish
// (atomic ticket, no waiting) merges the partials by log-sum-exp.
#include <cudaTypedefs.h>

#include <cmath>
#include <mutex>

#include "common.h"
#include "ptx.cuh"

namespace rgd {
namespace {

constexpr int kPage = 16;
constexpr int kCWarps = 15;                  // consumer warps (16 warps in all: <= 128 registers each)
constexpr int kCThreads = kCWarps * 32;
constexpr int kAttnThreads = kCThreads + 32;  // + one producer warp
constexpr int kMaxStages = 16;
constexpr int kMaxQueries = 128;  // rows_per_group * Hq / Hkv
constexpr int kSmemLimit = 226 * 1024;  // dynamic part; the kernel's static shared memory needs the rest
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
  float* slot_o;    // [(C + J - 1) * nq, D]
  float2* slot_ml;  // [(C + J - 1) * nq]
  int32_t* ticket;  // [J]
  int32_t* dev_status;
  int32_t G, rpg, Hq, Hkv, gq, num_pages, max_pp, max_sp;
  int32_t nq, n_mt, TS, nst, C;
  float scale_log2;
};

// Shared-memory carve-up (identical on host and device).
struct SmemLayout {
  int ring, q, acc, ml, gpre, desc, total;
};

__host__ __device__ inline int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <int D>
__host__ __device__ inline SmemLayout smem_layout(int nst, int n_mt, int TS, int G) {
  SmemLayout L;
  L.ring = 0;
  L.q = nst * 2 * kPage * D * 2;
  L.acc = align_up(L.q + n_mt * 16 * (D * 2 + 16), 16);
  L.ml = align_up(L.acc + n_mt * 16 * (D + 4) * 4, 16);
  L.gpre = align_up(L.ml + TS * n_mt * 16 * 8, 16);
  L.desc = align_up(L.gpre + (G + 1) * 4, 16);
  L.total = align_up(L.desc + nst * 4, 16) + 1024;  // + alignment slack for the 1024-B ring base
  return L;
}

// Byte offset of (token t, 16-byte chunk c) in a page tile loaded as 64-column
// boxes with the 128-byte swizzle (chunk index XOR row index mod 8).
__device__ __forceinline__ uint32_t swz(uint32_t tile, int t, int c) {
  return tile + ((c >> 3) << 11) + (t << 7) + ((((c & 7) ^ (t & 7))) << 4);
}

__device__ __forceinline__ void flag(int32_t* status, int32_t bit) {
  if (status) atomicOr(status, bit);
}

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kCThreads) : "memory"); }

__device__ __forceinline__ bool row_on(const AttnParams& p, int r) {
  return p.row_active == nullptr || p.row_active[r] != 0;
}

__device__ __forceinline__ int clamp_len(int n, int max_pages) { return n < 0 ? 0 : min(n, max_pages * kPage); }

// Pages of one (group, kv head) job: the prompt pages if any row of the group is
// active, plus the suffix pages of every active row.
__device__ int group_pages(const AttnParams& p, int g) {
  bool any = false;
  int sp = 0;
  for (int i = 0; i < p.rpg; ++i) {
    const int r = g * p.rpg + i;
    if (!row_on(p, r)) continue;
    any = true;
    sp += (clamp_len(p.suffix_len[r], p.max_sp) + kPage - 1) / kPage;
  }
  return any ? (clamp_len(p.prompt_len[g], p.max_pp) + kPage - 1) / kPage + sp : 0;
}

struct Job {
  int g, h, n;      // group, kv head, pages
  int64_t start;    // first page in the global page order
};

// The job containing global page x (x < total pages).
__device__ Job job_at(const AttnParams& p, const int32_t* gpre, int64_t x) {
  int lo = 0, hi = p.G - 1;  // largest g with Hkv * gpre[g] <= x
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if ((int64_t)p.Hkv * gpre[mid] <= x) lo = mid;
    else hi = mid - 1;
  }
  Job j;
  j.g = lo;
  j.n = gpre[lo + 1] - gpre[lo];
  const int64_t base = (int64_t)p.Hkv * gpre[lo];
  j.h = (int)((x - base) / j.n);
  j.start = base + (int64_t)j.h * j.n;
  return j;
}

__device__ Job next_job(const AttnParams& p, const int32_t* gpre, Job j) {
  j.start += j.n;
  if (++j.h == p.Hkv) {
    j.h = 0;
    do {
      ++j.g;
    } while (j.g < p.G && gpre[j.g + 1] == gpre[j.g]);
    j.n = j.g < p.G ? gpre[j.g + 1] - gpre[j.g] : 0;
    j.start = j.g < p.G ? (int64_t)p.Hkv * gpre[j.g] : j.start;
  }
  return j;
}

// CTA whose page range contains global page x (ranges [floor(cT/C), floor((c+1)T/C))).
__device__ __forceinline__ int cta_of(int64_t x, int64_t T, int C) { return (int)(((x + 1) * C - 1) / T); }

template <int D>
__global__ void __launch_bounds__(kAttnThreads, 1)
    attn_persistent_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                           const AttnParams p) {
  constexpr int kTile = kPage * D * 2;
  constexpr int kStage = 2 * kTile;
  constexpr int kQStride = D * 2 + 16;
  constexpr int kAccStride = D + 4;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SmemLayout L = smem_layout<D>(p.nst, p.n_mt, p.TS, p.G);
  int32_t* gpre = reinterpret_cast<int32_t*>(smem + L.gpre);
  uint32_t* descs = reinterpret_cast<uint32_t*>(smem + L.desc);
  uint8_t* qs = smem + L.q;
  float* acc = reinterpret_cast<float*>(smem + L.acc);
  float2* mls = reinterpret_cast<float2*>(smem + L.ml);
  __shared__ uint64_t full_bar[kMaxStages], empty_bar[kMaxStages];
  __shared__ int32_t s_abort, s_piece_abort, s_issued, s_last, s_wsum[kAttnThreads / 32];

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c = blockIdx.x;
  const int nst = p.nst;

  if (tid == 0) {
    for (int i = 0; i < nst; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], p.n_mt);
    }
    s_abort = 0;
    s_issued = 0;
    fence_mbar_init();
  }
  // ---- page counts per group and their exclusive prefix sum (every CTA) ----
  for (int g = tid; g < p.G; g += kAttnThreads) gpre[g + 1] = group_pages(p, g);
  if (tid == 0) gpre[0] = 0;
  if (c == 0) {
    for (int g = tid; g < p.G; g += kAttnThreads)
      if (p.prompt_len[g] < 0 || p.prompt_len[g] > p.max_pp * kPage) flag(p.dev_status, RGD_DEV_BAD_PAGE);
    for (int r = tid; r < p.G * p.rpg; r += kAttnThreads)
      if (p.suffix_len[r] < 0 || p.suffix_len[r] > p.max_sp * kPage) flag(p.dev_status, RGD_DEV_BAD_PAGE);
  }
  __syncthreads();
  {
    const int E = (p.G + kAttnThreads - 1) / kAttnThreads;
    const int lo = 1 + tid * E, hi = min(p.G + 1, lo + E);
    int sum = 0;
    for (int i = lo; i < hi; ++i) sum += gpre[i];
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) s_wsum[warp] = incl;
    __syncthreads();
    if (tid == 0) {
      int run = 0;
      for (int w = 0; w < kAttnThreads / 32; ++w) {
        const int t = s_wsum[w];
        s_wsum[w] = run;
        run += t;
      }
    }
    __syncthreads();
    int run = s_wsum[warp] + incl - sum;
    for (int i = lo; i < hi; ++i) {
      run += gpre[i];
      gpre[i] = run;
    }
  }
  __syncthreads();
  const int64_t T = (int64_t)p.Hkv * gpre[p.G];
  // pages are divided over Ceff = min(C, T) blocks so that every working block
  // has at least one page (a job's pieces are then exactly the blocks first..last)
  const int Ceff = (int)min((int64_t)p.C, T);
  const int64_t b = c < Ceff ? (int64_t)c * T / Ceff : T;
  const int64_t e = c < Ceff ? (int64_t)(c + 1) * T / Ceff : T;

  if (warp == kCWarps) {
    // ============================ producer ============================
    // The warp resolves 32 pages at a time, one per lane (job by binary search
    // in shared memory, then the block-table entry), so the global-memory
    // latency of the page lookups is paid once per 32 pages, and every lane then
    // issues its own page's two 4 KiB copies: the copy rate of a single issuing
    // thread, not HBM, is what limits a one-thread producer.
    if (b < e) {
      if (lane == 0) {
        prefetch_tensormap(&tmK);
        prefetch_tensormap(&tmV);
      }
      const uint64_t pol = policy_evict_first();
      bool aborted = false;
      // A batch holds at most one page per ring slot, so each lane's parity wait
      // on its slot is never more than one phase ahead of the consumers.
      const int nb = min(32, nst);
      for (int64_t xb = b; xb < e && !aborted; xb += nb) {
        const int64_t x = xb + lane;
        const bool mine = lane < nb && x < e;
        int32_t page = -1, tok = 0, rowsel = -1, hh = 0;
        if (mine) {
          const Job jb = job_at(p, gpre, x);
          const int k = (int)(x - jb.start);
          const int plen = clamp_len(p.prompt_len[jb.g], p.max_pp);
          const int ppg = (plen + kPage - 1) / kPage;
          hh = jb.h;
          if (k < ppg) {
            page = __ldg(p.prompt_bt + (int64_t)jb.g * p.max_pp + k);
            tok = min(kPage, plen - k * kPage);
          } else {
            int ks = k - ppg;
            for (int rr = 0; rr < p.rpg; ++rr) {  // the active row holding suffix page ks
              const int r = jb.g * p.rpg + rr;
              const int slen = row_on(p, r) ? clamp_len(p.suffix_len[r], p.max_sp) : 0;
              const int np = (slen + kPage - 1) / kPage;
              if (ks < np) {
                page = __ldg(p.suffix_bt + (int64_t)r * p.max_sp + ks);
                tok = min(kPage, slen - ks * kPage);
                rowsel = rr;
                break;
              }
              ks -= np;
            }
          }
        }
        // every lane issues its own page: up to 32 copy streams in flight
        int stop = 0;
        if (mine) {
          const int64_t li = x - b;
          const int slot = (int)(li % nst);
          if (li >= nst && !mbar_wait(&empty_bar[slot], (uint32_t)((li / nst) - 1) & 1u)) s_abort = 1;
          if (*(volatile int32_t*)&s_abort) {
            stop = 1;
          } else {
            int32_t y = -2 * kPage;  // fully out of bounds: the TMA fills zeros
            if (page >= 0 && page < p.num_pages) y = (page * p.Hkv + hh) * kPage;
            else flag(p.dev_status, RGD_DEV_BAD_PAGE);
            descs[slot] = (uint32_t)tok | ((uint32_t)(rowsel & 0xffff) << 16);
            uint8_t* kt = smem + slot * kStage;
            mbar_arrive_expect_tx(&full_bar[slot], kStage);
            tma_load_3d_hint(kt, &tmK, &full_bar[slot], 0, y, 0, pol);
            tma_load_3d_hint(kt + kTile, &tmV, &full_bar[slot], 0, y, 0, pol);
            atomicMax(&s_issued, (int)(li + 1));
          }
        }
        aborted = __any_sync(0xffffffffu, stop != 0);
      }
    }
  } else {
    // ============================ consumers ===========================
    const int n_mt = p.n_mt, TS = p.TS, nq = p.nq, gq = p.gq;
    const int mt = warp % n_mt, ts = warp / n_mt;
    const bool busy = warp < n_mt * TS;
    const int col = 2 * (lane & 3);
    const int qi0 = mt * 16 + (lane >> 2), qi1 = qi0 + 8;
    const int rloc0 = qi0 < nq ? qi0 / gq : -2, rloc1 = qi1 < nq ? qi1 / gq : -2;
    const uint32_t ring = smem_u32(smem);

    // jobs with no pages at all (empty prompt and suffixes, some row active)
    for (int j = c; j < p.G * p.Hkv; j += p.C) {
      const int g = j / p.Hkv, h = j % p.Hkv;
      if (gpre[g + 1] != gpre[g]) continue;
      for (int idx = tid; idx < nq * D; idx += kCThreads) {
        const int i = idx / D, d = idx % D;
        const int r = g * p.rpg + i / gq, hq = h * gq + i % gq;
        if (!row_on(p, r)) continue;
        p.out[((int64_t)r * p.Hq + hq) * D + d] = __float2bfloat16(0.f);
        if (d == 0 && p.lse) p.lse[(int64_t)r * p.Hq + hq] = -INFINITY;
      }
    }

    float o[D / 8][4];
    Job cur;
    if (b < e) cur = job_at(p, gpre, b);
    int64_t x0 = b;
    while (x0 < e) {
      const int64_t pe = min(e, cur.start + cur.n);
      const int j = cur.g * p.Hkv + cur.h;
      // ---- queries of the job -> shared memory; zero the combine buffer ----
      constexpr int kChunks = D / 8;
      for (int idx = tid; idx < n_mt * 16 * kChunks; idx += kCThreads) {
        const int i = idx / kChunks, ch = idx % kChunks;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (i < nq) {
          const int r = cur.g * p.rpg + i / gq, hq = cur.h * gq + i % gq;
          v = __ldg(reinterpret_cast<const uint4*>(p.q + ((int64_t)r * p.Hq + hq) * D) + ch);
        }
        *reinterpret_cast<uint4*>(qs + i * kQStride + ch * 16) = v;
      }
      for (int idx = tid; idx < n_mt * 16 * kAccStride; idx += kCThreads) acc[idx] = 0.f;
      consumer_sync();

      float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
#pragma unroll
      for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
      if (busy) {
        const uint32_t qbase =
            smem_u32(qs) + (mt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * kQStride + (lane >> 4) * 16;
        const int kt_t = (lane & 7) + ((lane >> 4) & 1) * 8, kt_c = (lane >> 3) & 1;
        const int vt_t = (lane & 7) + ((lane >> 3) & 1) * 8, vt_c = lane >> 4;
        const int lb = (int)(x0 - b), le = (int)(pe - b);
        int li = lb + ((ts - lb % TS) + TS) % TS;
        int slot = li % nst;  // ring slot and phase advance incrementally (TS divides nst)
        uint32_t phase = (uint32_t)(li / nst) & 1u;
        for (; li < le; li += TS) {
          if (*(volatile int32_t*)&s_abort) break;
          if (!mbar_wait(&full_bar[slot], phase)) {
            s_abort = 1;
            break;
          }
          const uint32_t desc = descs[slot];
          const int tok = (int)(desc & 0xffffu);
          const int rowsel = (int)(int16_t)(desc >> 16);
          const bool ok0 = rowsel < 0 || rloc0 == rowsel, ok1 = rowsel < 0 || rloc1 == rowsel;
          const uint32_t ktile = ring + slot * kStage, vtile = ktile + kTile;
          float sc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            uint32_t a[4], bq[4];
            ldmatrix_x4(a, qbase + kk * 32);
            ldmatrix_x4(bq, swz(ktile, kt_t, 2 * kk + kt_c));
            mma_bf16_16x8x16(sc[0], a, bq[0], bq[1]);
            mma_bf16_16x8x16(sc[1], a, bq[2], bq[3]);
          }
#pragma unroll
          for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int ee = 0; ee < 4; ++ee) {
              const int t = nt * 8 + col + (ee & 1);
              const bool ok = (t < tok) && (ee < 2 ? ok0 : ok1);
              sc[nt][ee] = ok ? sc[nt][ee] * p.scale_log2 : -INFINITY;
            }
          float mx0 = fmaxf(fmaxf(sc[0][0], sc[0][1]), fmaxf(sc[1][0], sc[1][1]));
          float mx1 = fmaxf(fmaxf(sc[0][2], sc[0][3]), fmaxf(sc[1][2], sc[1][3]));
          mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
          mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
          mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
          mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
          const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
          if (__any_sync(0xffffffffu, n0 != m0 || n1 != m1)) {
            // the running max moved for some row of the tile: rescale
            const float al0 = (n0 == m0) ? 1.f : exp2f(m0 - n0);
            const float al1 = (n1 == m1) ? 1.f : exp2f(m1 - n1);
            l0 *= al0;
            l1 *= al1;
#pragma unroll
            for (int i = 0; i < D / 8; ++i) {
              o[i][0] *= al0;
              o[i][1] *= al0;
              o[i][2] *= al1;
              o[i][3] *= al1;
            }
            m0 = n0;
            m1 = n1;
          }
          const float r0 = (m0 == -INFINITY) ? 0.f : m0, r1 = (m1 == -INFINITY) ? 0.f : m1;
          float pr[2][4];
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) {
            pr[nt][0] = exp2f(sc[nt][0] - r0);
            pr[nt][1] = exp2f(sc[nt][1] - r0);
            pr[nt][2] = exp2f(sc[nt][2] - r1);
            pr[nt][3] = exp2f(sc[nt][3] - r1);
          }
          l0 += (pr[0][0] + pr[0][1]) + (pr[1][0] + pr[1][1]);
          l1 += (pr[0][2] + pr[0][3]) + (pr[1][2] + pr[1][3]);
          uint32_t pa[4];
          pa[0] = pack_bf16x2(pr[0][0], pr[0][1]);
          pa[1] = pack_bf16x2(pr[0][2], pr[0][3]);
          pa[2] = pack_bf16x2(pr[1][0], pr[1][1]);
          pa[3] = pack_bf16x2(pr[1][2], pr[1][3]);
#pragma unroll
          for (int np = 0; np < D / 16; ++np) {
            uint32_t bv[4];
            ldmatrix_x4_trans(bv, swz(vtile, vt_t, 2 * np + vt_c));
            mma_bf16_16x8x16(o[2 * np], pa, bv[0], bv[1]);
            mma_bf16_16x8x16(o[2 * np + 1], pa, bv[2], bv[3]);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&empty_bar[slot]);
          slot += TS;
          if (slot >= nst) {
            slot -= nst;
            phase ^= 1u;
          }
        }
        l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
        l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
        l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
        if ((lane & 3) == 0) {
          mls[(ts * n_mt + mt) * 16 + (lane >> 2)] = make_float2(m0, l0);
          mls[(ts * n_mt + mt) * 16 + (lane >> 2) + 8] = make_float2(m1, l1);
        }
      }
      consumer_sync();
      // ---- combine the token slices: O = sum_t 2^(m_t - M) O_t --------------
      if (busy) {
        float M0 = -INFINITY, M1 = -INFINITY;
        for (int t = 0; t < TS; ++t) {
          M0 = fmaxf(M0, mls[(t * n_mt + mt) * 16 + (lane >> 2)].x);
          M1 = fmaxf(M1, mls[(t * n_mt + mt) * 16 + (lane >> 2) + 8].x);
        }
        const float f0 = (m0 == -INFINITY) ? 0.f : exp2f(m0 - M0);
        const float f1 = (m1 == -INFINITY) ? 0.f : exp2f(m1 - M1);
        float* a0 = acc + (mt * 16 + (lane >> 2)) * kAccStride + col;
        float* a1 = a0 + 8 * kAccStride;
        if (f0 != 0.f) {
#pragma unroll
          for (int i = 0; i < D / 8; ++i) {
            atomicAdd(a0 + i * 8, f0 * o[i][0]);
            atomicAdd(a0 + i * 8 + 1, f0 * o[i][1]);
          }
        }
        if (f1 != 0.f) {
#pragma unroll
          for (int i = 0; i < D / 8; ++i) {
            atomicAdd(a1 + i * 8, f1 * o[i][2]);
            atomicAdd(a1 + i * 8 + 1, f1 * o[i][3]);
          }
        }
      }
      // one thread snapshots the abort flag (the producer may set it at any time)
      // so that every consumer takes the same branch below
      if (tid == 0) s_piece_abort = *(volatile int32_t*)&s_abort;
      consumer_sync();
      const bool aborted = s_piece_abort != 0;
      const int first = cta_of(cur.start, T, Ceff), last = cta_of(cur.start + cur.n - 1, T, Ceff);
      // (M, L) of query i of this piece from the token-slice states
      auto piece_ml = [&](int i) {
        const int pm = i >> 4, pr = i & 15;
        float M = -INFINITY;
        for (int t = 0; t < TS; ++t) M = fmaxf(M, mls[(t * n_mt + pm) * 16 + pr].x);
        float Ls = 0.f;
        if (M != -INFINITY)
          for (int t = 0; t < TS; ++t) {
            const float2 v = mls[(t * n_mt + pm) * 16 + pr];
            Ls += v.y * exp2f(v.x - M);
          }
        return make_float2(M, Ls);
      };
      if (!aborted && first == last) {
        // the whole job is in this CTA: normalise and write the output
        for (int idx = tid; idx < nq * (D / 2); idx += kCThreads) {
          const int i = idx / (D / 2), d = 2 * (idx % (D / 2));
          const int r = cur.g * p.rpg + i / gq, hq = cur.h * gq + i % gq;
          if (!row_on(p, r)) continue;
          const float2 ml = piece_ml(i);
          const float inv = ml.y > 0.f ? 1.f / ml.y : 0.f;
          const float* a = acc + i * kAccStride + d;
          *reinterpret_cast<uint32_t*>(p.out + ((int64_t)r * p.Hq + hq) * D + d) =
              pack_bf16x2(a[0] * inv, a[1] * inv);
          if (d == 0 && p.lse)
            p.lse[(int64_t)r * p.Hq + hq] = ml.y > 0.f ? (ml.x + log2f(ml.y)) * kLn2 : -INFINITY;
        }
      } else if (!aborted) {
        // partial of a split job -> slot (cta + job); the last piece merges
        const int64_t s = (int64_t)c + j;
        for (int idx = tid; idx < nq * (D / 4); idx += kCThreads) {
          const int i = idx / (D / 4), d = 4 * (idx % (D / 4));
          const float* a = acc + i * kAccStride + d;
          *reinterpret_cast<float4*>(p.slot_o + (s * nq + i) * D + d) = make_float4(a[0], a[1], a[2], a[3]);
          if (d == 0) p.slot_ml[s * nq + i] = piece_ml(i);
        }
        __threadfence();
        consumer_sync();
        if (tid == 0) {
          const int prev = atomicAdd(p.ticket + j, 1);
          s_last = (prev == last - first);
          if (s_last) __threadfence();
        }
        consumer_sync();
        if (s_last) {
          constexpr int kPer = D / 32;
          for (int i = warp; i < nq; i += kCWarps) {
            const int r = cur.g * p.rpg + i / gq, hq = cur.h * gq + i % gq;
            if (!row_on(p, r)) continue;
            float M = -INFINITY;
            for (int cc = first; cc <= last; ++cc)
              M = fmaxf(M, __ldcg(&p.slot_ml[((int64_t)cc + j) * nq + i].x));
            float accv[kPer];
#pragma unroll
            for (int t = 0; t < kPer; ++t) accv[t] = 0.f;
            float Ls = 0.f;
            if (M != -INFINITY) {
              for (int cc = first; cc <= last; ++cc) {
                const int64_t si = ((int64_t)cc + j) * nq + i;
                const float2 ml = __ldcg(&p.slot_ml[si]);
                if (ml.y == 0.f) continue;
                const float w = exp2f(ml.x - M);
                Ls += w * ml.y;
                const float* po = p.slot_o + si * D + lane * kPer;
                if constexpr (kPer == 4) {
                  const float4 v = __ldcg(reinterpret_cast<const float4*>(po));
                  accv[0] += w * v.x;
                  accv[1] += w * v.y;
                  accv[2] += w * v.z;
                  accv[3] += w * v.w;
                } else {
                  const float2 v = __ldcg(reinterpret_cast<const float2*>(po));
                  accv[0] += w * v.x;
                  accv[1] += w * v.y;
                }
              }
            }
            const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
            __nv_bfloat16* dst = p.out + ((int64_t)r * p.Hq + hq) * D + lane * kPer;
            if constexpr (kPer == 4) {
              uint2 pk;
              pk.x = pack_bf16x2(accv[0] * inv, accv[1] * inv);
              pk.y = pack_bf16x2(accv[2] * inv, accv[3] * inv);
              *reinterpret_cast<uint2*>(dst) = pk;
            } else {
              *reinterpret_cast<uint32_t*>(dst) = pack_bf16x2(accv[0] * inv, accv[1] * inv);
            }
            if (p.lse && lane == 0)
              p.lse[(int64_t)r * p.Hq + hq] = Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY;
          }
          if (tid == 0) p.ticket[j] = 0;
        }
      }
      consumer_sync();  // Q, acc and the slice states are reused by the next piece
      x0 = pe;
      if (x0 < e) cur = next_job(p, gpre, cur);
    }
  }
  __syncthreads();
  if (s_abort && tid == 0) {
    // a copy did not land: report, and wait (bounded) for the copies still in flight
    flag(p.dev_status, RGD_DEV_WAIT_TIMEOUT);
    for (int li = max(0, s_issued - nst); li < s_issued; ++li) mbar_wait(&full_bar[li % nst], (li / nst) & 1);
  }
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
  // View each 16-token page-head tile as (64 columns) x (16 rows) x (D/64 halves):
  // one box is the whole tile, laid out in shared memory half-major with the
  // 128-byte swizzle (16-byte chunk index XOR row index mod 8).
  cuuint64_t dims[3] = {64, (cuuint64_t)rows, (cuuint64_t)(D / 64)};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, 128};
  cuuint32_t box[3] = {64, (cuuint32_t)kPage, (cuuint32_t)(D / 64)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_error(RGD_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return RGD_OK;
}

int device_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

struct Plan {
  int nq, n_mt, TS, nst, C, J;
  SmemLayout smem;
  size_t ticket_off, ml_off, o_off, total;
};

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
  RGD_CHECK_ARG(s->num_ctas >= 0 && s->reserved == 0, "num_ctas must be >= 0 and reserved 0");
  RGD_CHECK_ARG((int64_t)s->num_groups * (s->max_prompt_pages + (int64_t)s->rows_per_group * s->max_suffix_pages) *
                        s->num_kv_heads <
                    ((int64_t)1 << 31),
                "too many KV pages in one call (must be < 2^31)");
  const int nq = s->rows_per_group * (s->num_q_heads / s->num_kv_heads);
  if (nq > kMaxQueries)
    return set_error(RGD_ERR_UNSUPPORTED, "rows_per_group * Hq/Hkv = %d exceeds %d", nq, kMaxQueries);
  return RGD_OK;
}

int make_plan(const rgd_attn_shape* s, Plan* pl) {
  if (int rc = check_shape(s)) return rc;
  pl->nq = s->rows_per_group * (s->num_q_heads / s->num_kv_heads);
  pl->n_mt = (pl->nq + 15) / 16;
  pl->TS = kCWarps / pl->n_mt;
  pl->C = s->num_ctas > 0 ? s->num_ctas : device_sm_count();
  if (pl->C <= 0) return set_error(RGD_ERR_CUDA, "could not query the device's SM count");
  pl->J = s->num_groups * s->num_kv_heads;
  pl->nst = (kMaxStages / pl->TS) * pl->TS;
  for (;;) {
    pl->smem = s->head_dim == 128 ? smem_layout<128>(pl->nst, pl->n_mt, pl->TS, s->num_groups)
                                  : smem_layout<64>(pl->nst, pl->n_mt, pl->TS, s->num_groups);
    if (pl->smem.total <= kSmemLimit) break;
    if (pl->nst <= pl->TS)
      return set_error(RGD_ERR_UNSUPPORTED, "shape needs more shared memory than an SM has (too many groups?)");
    pl->nst -= pl->TS;
  }
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  const size_t nslots = (size_t)pl->C + pl->J - 1;
  pl->ticket_off = 0;
  pl->ml_off = up((size_t)pl->J * sizeof(int32_t));
  pl->o_off = pl->ml_off + up(nslots * pl->nq * sizeof(float2));
  pl->total = pl->o_off + up(nslots * pl->nq * s->head_dim * sizeof(float));
  return RGD_OK;
}

// Workspace fields used by the allocation-free entry point below.
struct WsLayout {
  size_t ml_off, total;
};

WsLayout ws_layout(const rgd_attn_shape* s) {
  Plan pl;
  WsLayout w{0, 0};
  if (make_plan(s, &pl) == RGD_OK) {
    w.ml_off = pl.ml_off;
    w.total = pl.total;
  }
  return w;
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" size_t rgd_prefix_decode_attn_workspace_size(const rgd_attn_shape* shape) {
  clear_error();
  Plan pl;
  if (make_plan(shape, &pl) != RGD_OK) return 0;
  return pl.total;
}

extern "C" int rgd_prefix_decode_attn(const rgd_attn_shape* shape, const rgd_bf16* q, const rgd_bf16* k_pages,
                                      const rgd_bf16* v_pages, const int32_t* prompt_block_table,
                                      const int32_t* prompt_len, const int32_t* suffix_block_table,
                                      const int32_t* suffix_len, const uint8_t* row_active, float softmax_scale,
                                      rgd_bf16* out, float* lse, void* workspace, size_t workspace_bytes,
                                      int32_t* dev_status, rgd_stream_t stream) {
  clear_error();
  Plan pl;
  if (int rc = make_plan(shape, &pl)) return rc;
  const rgd_attn_shape& s = *shape;
  RGD_CHECK_ARG(q && k_pages && v_pages && prompt_block_table && prompt_len && suffix_block_table && suffix_len &&
                    out && workspace,
                "rgd_prefix_decode_attn: a required pointer is NULL");
  RGD_CHECK_ARG(aligned16(q) && aligned16(k_pages) && aligned16(v_pages) && aligned16(out),
                "rgd_prefix_decode_attn: q, k_pages, v_pages and out must be 16-byte aligned");
  RGD_CHECK_ARG((reinterpret_cast<uintptr_t>(workspace) & 255) == 0, "workspace must be 256-byte aligned");
  RGD_CHECK_ARG(std::isfinite(softmax_scale) && softmax_scale > 0.f, "softmax_scale must be > 0");
  RGD_CHECK_ARG(workspace_bytes >= pl.total, "workspace too small: %zu < %zu", workspace_bytes, pl.total);

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
  p.ticket = reinterpret_cast<int32_t*>(ws + pl.ticket_off);
  p.slot_ml = reinterpret_cast<float2*>(ws + pl.ml_off);
  p.slot_o = reinterpret_cast<float*>(ws + pl.o_off);
  p.dev_status = dev_status;
  p.G = s.num_groups;
  p.rpg = s.rows_per_group;
  p.Hq = s.num_q_heads;
  p.Hkv = s.num_kv_heads;
  p.gq = s.num_q_heads / s.num_kv_heads;
  p.num_pages = s.num_pages;
  p.max_pp = s.max_prompt_pages;
  p.max_sp = s.max_suffix_pages;
  p.nq = pl.nq;
  p.n_mt = pl.n_mt;
  p.TS = pl.TS;
  p.nst = pl.nst;
  p.C = pl.C;
  p.scale_log2 = softmax_scale * kLog2e;

  cudaStream_t st = (cudaStream_t)stream;
  if (s.head_dim == 128) {
    static bool done = false;
    if (int rc = ensure_smem(attn_persistent_kernel<128>, kSmemLimit, &done)) return rc;
    attn_persistent_kernel<128><<<pl.C, kAttnThreads, pl.smem.total, st>>>(tmK, tmV, p);
  } else {
    static bool done = false;
    if (int rc = ensure_smem(attn_persistent_kernel<64>, kSmemLimit, &done)) return rc;
    attn_persistent_kernel<64><<<pl.C, kAttnThreads, pl.smem.total, st>>>(tmK, tmV, p);
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
