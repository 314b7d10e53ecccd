// Shared-prefix decode attention on the 5th-generation tensor cores.
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
// the grid's persistent blocks (one per SM) each take an equal contiguous range
// of pages.  Only the two jobs at the ends of a block's range can be split with
// a neighbour, and a block works on those two first (the end of the job it
// starts in, then the start of the job it ends in, then the whole jobs between).
// A split job is merged by log-sum-exp (Sec. 3's shared-prefix split is the same
// identity) in the block holding its first page: the job's other pieces --
// each the first piece of its own block -- write a partial (o, m, l) to
// workspace slot (block + job) and count themselves in the job's ticket; the
// merger's watcher warp polls the ticket while its own piece runs, brings the
// partials into shared memory by bulk copies once all have counted, and folds
// them into its own O on the way out.
//
// Inside a block (384 threads for R = 4 query copies, 512 for 2, 640 for 1) the
// tensor memory holds Q, S, P and O, so the tensor cores read only K and V from
// shared memory -- the bytes that come from HBM:
//   * two producer warps take alternate rounds of 32 pages and stream them,
//     four to a group, into a ring of group slots with 3-D TMA boxes (128-byte
//     swizzle): each K tile lands as two 2 KiB halves in a half-major,
//     group-contiguous block, so that one MMA covers all the group's tokens (an
//     MMA costs ~50 cycles to issue whatever its N, so the number of MMAs, not
//     their size, is what counts), each V tile as one box; every lane issues
//     its own page, since one issuing thread is copy-rate bound;
//   * the QK warp allocates the tensor memory and its lane 0 issues, per group
//     of up to 4 pages, S = Q K^T (A = Q from TMEM, M = 128 query rows,
//     N = 16 x pages) into the S buffer; the softmax warps turn S into P (a
//     bf16 high part and a bf16 residual, in two P buffers), and lane 0 of the
//     PV warp issues O += P V for both parts per page (A = P from TMEM, N = the
//     head dimension, V read MN-major from its tile); one commit after the
//     group's PV hands its slot back to the producers;
//   * softmax warps: warp w can reach TMEM lanes 32(w%4)..+31 only.  The job's
//     queries are held in R copies in the 128 lanes; a softmax warp handles the
//     16 scores of one page for 32 query rows of one copy: the masks, the row
//     max (shared through shared memory by the warps of a copy that share
//     rows), the online softmax in fp32 (the running max is only moved, and O
//     rescaled in TMEM, when a row's max grows by more than 2^8) and its P;
//   * epilogue warps (one per used lane quarter when R > 1; the softmax warps
//     themselves when R = 1) write the next piece's Q into TMEM once the
//     current piece's last QK is done, and at a piece's end read O (double-
//     buffered by piece, so the softmax warps go on meanwhile), merge the copies
//     by log-sum-exp through shared memory and write the output, the partial
//     of a split job, or -- in a merger -- the merged output.
// Every wait on an mbarrier is bounded; a timeout is reported in the status
// word and every role stops.
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <mutex>

#include "common.h"
#include "ptx.cuh"

namespace rgd {
namespace {

constexpr int kPage = 16;
constexpr int kProducerWarps = 2;

// Warp roles of the attention kernel for R copies of the job's queries in the
// 128 TMEM lanes (R = 4 / the lane quarters one copy spans).  Each used lane
// quarter gets W = 4 / R softmax warps (one page of a group each) and, when
// R > 1, one epilogue warp; then come two producers, the QK issuer and the PV
// issuer.  Fewer warps leave each more registers (384 threads at R = 4).
template <int R>
struct Roles {
  static constexpr int kW = 4 / R;                   // softmax warps per quarter
  static constexpr int kNE = R > 1 ? 1 : 0;          // spare epilogue warps per quarter
  static constexpr int kSoft = 4 * (kW + kNE);       // softmax and epilogue warps
  static constexpr int kProducer = kSoft;            // kProducerWarps page producers
  static constexpr int kMma = kSoft + kProducerWarps;  // QK issue (and the TMEM allocation)
  static constexpr int kPv = kMma + 1;               // PV issue
  static constexpr int kThreads = (kPv + 1) * 32;
};
constexpr int kMaxAttnWarps = Roles<1>::kThreads / 32;
constexpr int kGroupPages = 4;                // pages per S / P buffer (64 tokens)
constexpr int kMaxSlots = 8;                  // ring slots, one page group each
constexpr int kSBufs = 1;                     // S buffers in TMEM (freed once the softmax has read them)
constexpr int kPBufs = 2;                     // P buffers in TMEM (freed once their PV is done)
constexpr int kRows = 128;                    // MMA M: query rows per job
constexpr int kMaxQueries = kRows;            // rows_per_group * Hq / Hkv
constexpr int kTmemCols = 512;
constexpr int kOCol = 0;                      // O: two buffers (alternate job pieces) of D columns
constexpr int kOStride = 128;
constexpr int kSCol = 2 * kOStride;           // S buffers: 64 fp32 columns each (4 pages x 16 tokens)
constexpr int kPCol = kSCol + kSBufs * 64;    // P buffers: 32 columns each (4 pages x 16 bf16), high parts
constexpr int kPLoCol = kPCol + kPBufs * 32;  // the matching bf16 residuals P - bf16(P)
constexpr int kQCol = kPLoCol + kPBufs * 32;  // Q: D/2 columns (two bf16 per column)
static_assert(kQCol + 64 <= 512, "TMEM columns");
// V as the MN-major B operand of PV: the two 64-column halves of a page tile are
// MN-direction swizzle atoms 2048 B apart, the two 8-token groups K-direction
// atoms 1024 B apart.
constexpr uint32_t kVLbo = 2048, kVSbo = 1024;
constexpr float kRescaleLog2 = 8.f;           // lazy rescale threshold (factor 256)
constexpr int kSmemLimit = 226 * 1024;        // dynamic part; static shared memory needs the rest
constexpr int kTicketSlots = 8192;            // job counters at the start of every workspace (at least)
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
  float2* slot_ml;  // [(C + J - 1) * ml_stride(nq)]
  int32_t* ticket;  // [J] pieces of a split job that have finished (zero between calls)
  int npref;        // partner pieces whose partials fit the prefetch area (1 or 2)
  int32_t* dev_status;
  int32_t G, rpg, Hq, Hkv, gq, num_pages, max_pp, max_sp;
  int32_t nq, nslots, C;
  float scale_log2;
  uint64_t wait_ns;  // limit of every wait on another role or block (rgd_set_wait_limit_ns)
};

// Shared-memory carve-up (identical on host and device).  The ring is 1024-byte
// aligned: the 128-byte swizzle repeats every 8 rows of 128 bytes.
struct SmemLayout {
  int ring, red, gpre, plen, desc, rowbits, slen, pref, total;
};

// Partial (m, l) pairs are stored nq rounded up to even per piece, so that
// every piece's pairs start on a 16-byte boundary (bulk copies).
__host__ __device__ constexpr int ml_stride(int nq) { return (nq + 1) & ~1; }

// Shared memory for one partner piece's partial result, prefetched by the block
// that will merge a split job: O rows padded to D + 4 floats (conflict-free
// row-per-lane reads), then the (m, l) pairs.
template <int D>
__host__ __device__ constexpr int pref_bytes(int nq) { return nq * (D + 4) * 4 + ml_stride(nq) * 8; }

__host__ __device__ inline int align_up(int x, int a) { return (x + a - 1) / a * a; }

// One ring slot holds a page group: its K tiles half-major and group-contiguous
// ([D/64 halves][4 pages][16 rows][128 B], so that one MMA reads the whole
// group's K for a 16-wide slice of the head dimension), then its V tiles
// ([4 pages][D/64 halves][16 rows][128 B]).
template <int D>
__host__ __device__ constexpr int slot_bytes() {
  return 2 * kGroupPages * kPage * D * 2;
}

template <int D>
__host__ __device__ inline SmemLayout smem_layout(int nslots, int G, int R, int nq, int npref) {
  SmemLayout L;
  L.ring = 0;
  L.red = nslots * slot_bytes<D>();
  // row-max exchange (2 buffers), row sums and running maxima of 2 pieces, O
  // staging for the copies >= 1 (2 buffers of at most 3 warps x 16 columns x 32 lanes)
  L.gpre = L.red + (2 * 4 * kRows + 2 * 4 * kRows + 2 * kRows + 2 * 3 * 4 * 32 * 4) * 4;
  L.plen = align_up(L.gpre + (G + 1) * 4, 16);  // prompt length per group (clamped)
  L.desc = align_up(L.plen + G * 4, 16);
  L.rowbits = align_up(L.desc + nslots * kGroupPages * 4, 16);  // one bit per row: active
  L.slen = align_up(L.rowbits + (R + 31) / 32 * 4, 16);          // suffix length per row (0: inactive)
  L.pref = align_up(L.slen + R * 4, 16);
  L.total = L.pref + npref * pref_bytes<D>(nq) + 1024;  // + slack for the 1024-byte aligned base
  return L;
}

__device__ __forceinline__ void flag(int32_t* status, int32_t bit) {
  if (status) atomicOr(status, bit);
}

__device__ __forceinline__ bool row_on(const AttnParams& p, int r) {
  return p.row_active == nullptr || p.row_active[r] != 0;
}

__device__ __forceinline__ int clamp_len(int n, int max_pages) { return n < 0 ? 0 : min(n, max_pages * kPage); }

struct Job {
  int g, h, n;      // group, kv head, pages
  int64_t start;    // first page in the global page order
};

// The job containing global page x (x < total pages).
// a / b for a >= 0, b > 0: 32-bit division when both fit (the usual case;
// 64-bit division is a long instruction sequence on the GPU).
__device__ __forceinline__ int64_t div_nn(int64_t a, int64_t b) {
  if (((uint64_t)a | (uint64_t)b) >> 32 == 0) return (int64_t)((uint32_t)a / (uint32_t)b);
  return a / b;
}

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
  j.h = (int)div_nn(x - base, j.n);
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

// Block whose page range contains global page x (ranges [floor(cT/C), floor((c+1)T/C))).
__device__ __forceinline__ int cta_of(int64_t x, int64_t T, int C) { return (int)div_nn((x + 1) * C - 1, T); }

// A block's job pieces in the order it works on them: the job at the start of
// its range, then the job at the end, then the whole jobs in between.  Only the
// two end jobs can be split with a neighbouring block, so every split job is
// finished early in both of its blocks and is merged off their critical paths.
struct PieceIter {
  Job j0, jl;       // first and last job of the range
  int n0, nl;       // their pages in the range (nl = 0: the range holds one job)
  int64_t mid_end;  // global page where the middle jobs end
};

__device__ PieceIter piece_iter(const AttnParams& p, const int32_t* gpre, int64_t b, int64_t e) {
  PieceIter it;
  it.j0 = job_at(p, gpre, b);
  it.n0 = (int)(min(e, it.j0.start + it.j0.n) - b);
  it.jl = it.j0;
  it.nl = 0;
  it.mid_end = e;
  if (b + it.n0 < e) {
    it.jl = job_at(p, gpre, e - 1);
    it.nl = (int)(e - it.jl.start);
    it.mid_end = it.jl.start;
  }
  return it;
}

// Piece k (>= 1) after piece k - 1 = (cur, n); false when there is none.
__device__ bool next_piece(const AttnParams& p, const int32_t* gpre, const PieceIter& it, int k, Job& cur, int& n) {
  if (k == 1) {
    if (it.nl == 0) return false;
    cur = it.jl;
    n = it.nl;
    return true;
  }
  const Job nx = next_job(p, gpre, k == 2 ? it.j0 : cur);
  if (nx.start >= it.mid_end) return false;
  cur = nx;
  n = nx.n;
  return true;
}

// Global page of position i of a block's page sequence (pieces in PieceIter order).
__device__ __forceinline__ int64_t seq_page(const PieceIter& it, int64_t b, int64_t i) {
  if (i < it.n0) return b + i;
  if (i < it.n0 + it.nl) return it.jl.start + (i - it.n0);
  return b + it.n0 + (i - it.n0 - it.nl);
}

// Bounded wait that also gives up as soon as another role has given up.
// A waiting thread sleeps inside try_wait (woken when the phase completes), so
// warps parked on a barrier take no issue slots from the working ones.
__device__ __noinline__ bool wait_or_abort_slow(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag,
                                                uint64_t limit_ns) {
  if (*abort_flag) return false;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort_flag = 1;
        return false;
      }
    }
  }
}
// (the loop is out of line: it is only reached when the phase has not completed
// at the first look, and one copy keeps the kernels' code small)
__device__ __forceinline__ bool wait_or_abort(uint64_t* bar, uint32_t parity, volatile int32_t* abort_flag,
                                              uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  return wait_or_abort_slow(bar, parity, abort_flag, limit_ns);
}

// Bounded wait until *gen >= want (a shared counter another warp raises).
__device__ __forceinline__ bool wait_slot_gen(int32_t* gen, int32_t want, volatile int32_t* abort_flag,
                                              uint64_t limit_ns) {
  volatile int32_t* g = gen;
  if (*g >= want) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (*g >= want) return true;
    if ((i & 63u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort_flag = 1;
        return false;
      }
    }
    __nanosleep(32);
  }
}

// The merge of a split job whose other pieces' partials do not fit the
// prefetch area: every piece's partial read straight from global memory (L2,
// past L1) after the job's count is complete; each of the n_et epilogue
// threads folds its kU float4 columns of O over the pieces in order (the loads
// of one piece for all of them in flight at once) and writes the output.  Out
// of line, so that its registers do not crowd the kernel's other code.
template <int D>
__device__ __noinline__ void merge_from_l2(const float2* slot_ml, const float* slot_o, __nv_bfloat16* out, float* lse,
                                           int nq, int gq, int rpg, int Hq, int g, int h, int jj, int first,
                                           int last, int et, int n_et, const uint32_t* rowbits, bool good) {
  constexpr int kU = 4;  // columns per thread per pass
  const int mls = ml_stride(nq), n4 = nq * (D / 4);
  for (int b0 = 0; b0 < n4; b0 += kU * n_et) {
    const int base = b0 + et;
    float Mm[kU], Lm[kU];
    float4 acc[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      Mm[u] = -INFINITY;
      Lm[u] = 0.f;
      acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int s2 = first; s2 <= last && good; ++s2) {
      const int64_t sl = (int64_t)s2 + jj;
      float2 ml[kU];
      float4 v[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int it = base + u * n_et;
        ml[u] = make_float2(-INFINITY, 0.f);
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (it < n4) {
          const int i = it / (D / 4), c4 = it % (D / 4);
          ml[u] = __ldcg(slot_ml + sl * mls + i);
          v[u] = __ldcg(reinterpret_cast<const float4*>(slot_o + (sl * nq + i) * D) + c4);
        }
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        if (ml[u].y == 0.f) continue;
        const float Mn = fmaxf(Mm[u], ml[u].x);
        const float f = Mm[u] == -INFINITY ? 0.f : exp2f(Mm[u] - Mn), w = exp2f(ml[u].x - Mn);
        Lm[u] = Lm[u] * f + w * ml[u].y;
        acc[u].x = acc[u].x * f + w * v[u].x;
        acc[u].y = acc[u].y * f + w * v[u].y;
        acc[u].z = acc[u].z * f + w * v[u].z;
        acc[u].w = acc[u].w * f + w * v[u].w;
        Mm[u] = Mn;
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int it = base + u * n_et;
      if (!good || it >= n4) break;  // (after an abort the outputs are not written)
      const int i = it / (D / 4), c4 = it % (D / 4);
      const int rr2 = g * rpg + i / gq, hq2 = h * gq + i % gq;
      if (!((rowbits[rr2 >> 5] >> (rr2 & 31)) & 1u)) continue;
      const float iv = Lm[u] > 0.f ? 1.f / Lm[u] : 0.f;
      uint2 pk2;
      pk2.x = pack_bf16x2(acc[u].x * iv, acc[u].y * iv);
      pk2.y = pack_bf16x2(acc[u].z * iv, acc[u].w * iv);
      reinterpret_cast<uint2*>(out + ((int64_t)rr2 * Hq + hq2) * D)[c4] = pk2;
      if (lse && c4 == 0) lse[(int64_t)rr2 * Hq + hq2] = Lm[u] > 0.f ? (Mm[u] + log2f(Lm[u])) * kLn2 : -INFINITY;
    }
  }
}

template <int D, int R>
__global__ void __launch_bounds__(Roles<R>::kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const AttnParams p) {
  constexpr int kTile = kPage * D * 2;      // one K or V page-head tile
  constexpr int kStage = 2 * kTile;         // bytes one page brings in
  constexpr int kHalves = D / 64;
  constexpr int kSlot = slot_bytes<D>();
  constexpr int kVOff = kGroupPages * kTile;  // V tiles within a slot
  constexpr uint32_t kIdescPV = idesc_bf16_f32(kRows, D, 0, 1);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const SmemLayout L = smem_layout<D>(p.nslots, p.G, p.G * p.rpg, p.nq, p.npref);
  uint32_t* rowbits = reinterpret_cast<uint32_t*>(smem + L.rowbits);
  int32_t* gpre = reinterpret_cast<int32_t*>(smem + L.gpre);
  uint32_t* descs = reinterpret_cast<uint32_t*>(smem + L.desc);
  __shared__ uint64_t full_bar[kMaxSlots], empty_bar[kMaxSlots];
  __shared__ uint64_t s_full[kSBufs], s_empty[kSBufs], p_full[kPBufs], p_empty[kPBufs];
  __shared__ uint64_t q_full, q_empty, o_full[2], o_free[2], ml_full[2], ml_empty[2], mma_done[2];
  __shared__ uint64_t pref_bar;  // a split job's partner partials have landed in shared memory
  using Rl = Roles<R>;
  constexpr int kAttnThreads = Rl::kThreads;
  constexpr int kSoftThreads = Rl::kSoft * 32;
  constexpr int kProducerWarp = Rl::kProducer, kMmaWarp = Rl::kMma, kPvWarp = Rl::kPv;
  __shared__ int32_t s_abort, s_issued, s_last, s_pref_n, s_wsum[kMaxAttnWarps];
  __shared__ int32_t s_slot_gen[kMaxSlots];  // the last group that entered each ring slot
  __shared__ uint32_t s_tmem;
  volatile int32_t* abort_flag = &s_abort;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c = blockIdx.x;
  const int ns = p.nslots;
  const uint32_t sbase = smem_u32(smem);
  // The queries fill qpc TMEM lane quarters and are held R times; the softmax
  // warps of unused quarters sit out, and the barriers count the active ones.
  const int qpc = (p.nq + 31) / 32;         // lane quarters one copy of the queries spans (4 / R, or 3)
  constexpr int W = Rl::kW;                 // softmax warps per quarter (pages per copy and group)
  constexpr bool side = Rl::kNE > 0;        // a spare warp per quarter does the piece ends
  constexpr int NE = side ? Rl::kNE : W;    // epilogue (and Q-writing) warps per used quarter
  const int n_soft = R * qpc * W;           // softmax warps of each group
  const int n_epi = R * qpc * NE;           // warps that write Q and finish pieces

  if (tid == 0) {
    for (int i = 0; i < ns; ++i) {
      mbar_init(&full_bar[i], kGroupPages);  // one arrival per page position (absent pages of a short group too)
      mbar_init(&empty_bar[i], 1);           // released by an MMA commit once the group's PV is done
    }
    for (int i = 0; i < kSBufs; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], n_soft);
    }
    for (int i = 0; i < kPBufs; ++i) {
      mbar_init(&p_full[i], n_soft);
      mbar_init(&p_empty[i], 1);
    }
    mbar_init(&q_full, n_epi);
    mbar_init(&q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&o_full[i], 1);
      mbar_init(&o_free[i], n_epi);
      mbar_init(&ml_full[i], n_soft);
      mbar_init(&ml_empty[i], n_epi);
    }
    mbar_init(&mma_done[0], 1);
    mbar_init(&mma_done[1], 1);
    mbar_init(&pref_bar, 1);
    s_abort = 0;
    s_issued = 0;
    s_pref_n = 0;  // partner prefetches issued
    for (int i = 0; i < kMaxSlots; ++i) s_slot_gen[i] = -1;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&s_tmem, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kProducerWarp && lane == 0) {  // the copies' descriptors, fetched while the set-up runs
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
  }
  // ---- page counts per group and their exclusive prefix sum (every block) ----
  // The lengths and activity flags are read once, all loads issued together
  // (one global-memory latency), and kept in shared memory for the producer.
  int32_t* plen_s = reinterpret_cast<int32_t*>(smem + L.plen);
  int32_t* slen_s = reinterpret_cast<int32_t*>(smem + L.slen);
  const int nrows = p.G * p.rpg;
  for (int r0 = warp * 32; r0 < nrows; r0 += kAttnThreads) {  // (whole warps: the ballot below)
    const int r = r0 + lane;
    int act = 0, sl = 0;
    if (r < nrows) {
      act = p.row_active == nullptr ? 1 : p.row_active[r];
      sl = p.suffix_len[r];
      if (c == 0 && (sl < 0 || sl > p.max_sp * kPage)) flag(p.dev_status, RGD_DEV_BAD_PAGE);
      slen_s[r] = act ? clamp_len(sl, p.max_sp) : 0;
    }
    const uint32_t bits = __ballot_sync(0xffffffffu, r < nrows && act != 0);
    if (lane == 0) rowbits[r0 >> 5] = bits;
  }
  for (int g = tid; g < p.G; g += kAttnThreads) {
    const int pl = p.prompt_len[g];
    if (c == 0 && (pl < 0 || pl > p.max_pp * kPage)) flag(p.dev_status, RGD_DEV_BAD_PAGE);
    plen_s[g] = clamp_len(pl, p.max_pp);
  }
  if (tid == 0) gpre[0] = 0;
  __syncthreads();
  // a group's pages: its prompt pages if any row of it is active, plus its
  // active rows' suffix pages
  for (int g = tid; g < p.G; g += kAttnThreads) {
    int n = 0;
    bool any = false;
    for (int rr = 0; rr < p.rpg; ++rr) {
      const int r = g * p.rpg + rr;
      n += (slen_s[r] + kPage - 1) / kPage;
      any = any || ((rowbits[r >> 5] >> (r & 31)) & 1u);
    }
    gpre[g + 1] = any ? n + (plen_s[g] + kPage - 1) / kPage : 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
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
  const int64_t b = c < Ceff ? div_nn((int64_t)c * T, Ceff) : T;
  const int64_t e = c < Ceff ? div_nn((int64_t)(c + 1) * T, Ceff) : T;
  // the piece order, kept in shared memory (read at piece boundaries only)
  __shared__ PieceIter s_it;
  if (tid == 0 && b < e) s_it = piece_iter(p, gpre, b, e);
  __syncthreads();

  if (warp >= kProducerWarp && warp < kProducerWarp + kProducerWarps) {
    // ============================ producers ===========================
    // The block's pages are taken 32 at a time, one per lane; the two producer
    // warps take alternate rounds, so that one warp's block-table loads overlap
    // the other's copies, and each issues half the copies.  Both walk every
    // round to number the groups (group g of this block goes to slot
    // g % nslots; groups restart at each job piece), which needs only shared
    // memory.  In its own rounds a warp resolves each page (job by binary
    // search, then the block-table entry) and then, group by group, the first
    // lane of the group in the round waits for the slot and every lane of the
    // group issues its page's copies: K as two 2 KiB halves into the group's
    // half-major K block, V as one box.  A slot wait (for the PV of the group
    // nslots back, issued after the QK of the group after it) depends only on
    // pages of earlier groups, and a warp's waits in a round depend only on
    // pages of earlier rounds, so neither warp can hold up the other.
    const int pw = warp - kProducerWarp;
    if (b < e) {
      const uint64_t pol = policy_evict_first();
      const PieceIter& it = s_it;
      int gbase = 0;  // groups started before sequence position ib
      int rnd = 0;
      for (int64_t ib = 0; ib < e - b; ib += 32, ++rnd) {
        const bool valid = ib + lane < e - b;
        const int64_t x = valid ? seq_page(it, b, ib + lane) : b;
        const bool mine = (rnd % kProducerWarps) == pw;
        int32_t page = -1, tok = 0, rowsel = -1, hh = 0, jpos = 0, ng = 0;
        if (valid) {
          const Job jb = job_at(p, gpre, x);
          // this block's piece of the job starts at max(b, job start); groups restart there
          const int64_t pstart = max(b, jb.start);
          const int kin = (int)(x - pstart);
          const int npiece = (int)(min(e, jb.start + jb.n) - pstart);
          jpos = kin % kGroupPages;
          ng = min(kGroupPages, npiece - (kin - jpos));
          if (mine) {
            const int k = (int)(x - jb.start);
            const int plen = plen_s[jb.g];
            const int ppg = (plen + kPage - 1) / kPage;
            hh = jb.h;
            if (k < ppg) {
              page = __ldg(p.prompt_bt + (int64_t)jb.g * p.max_pp + k);
              tok = min(kPage, plen - k * kPage);
            } else {
              int ks = k - ppg;
              for (int rr = 0; rr < p.rpg; ++rr) {  // the active row holding suffix page ks
                const int r = jb.g * p.rpg + rr;
                const int slen = slen_s[r];
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
        }
        const bool start = valid && jpos == 0;
        const uint32_t starts = __ballot_sync(0xffffffffu, start);
        if (mine) {
          const uint32_t le = 0xffffffffu >> (31 - lane);
          const int gidx = gbase + __popc(starts & le) - 1;  // lane 0 may continue the last round's group
          const int g0 = __shfl_sync(0xffffffffu, gidx, 0);
          const int g1 = __shfl_sync(0xffffffffu, gidx, 31 - __clz(__ballot_sync(0xffffffffu, valid)));
          const int gs = gidx % ns;
          bool aborted = false;
          for (int gq = g0; gq <= g1; ++gq) {
            const bool in = valid && gidx == gq;
            // the group's first lane in this round waits for the slot: first until
            // the slot's previous group has entered it (the other warp may still be
            // behind), so that the parity wait on its release is never two phases
            // ahead, then for that release
            const bool lead = in && (start || lane == 0);
            int stop = 0;
            if (lead && gq >= ns &&
                (!wait_slot_gen(&s_slot_gen[gs], gq - ns, abort_flag, p.wait_ns) ||
                 !wait_or_abort(&empty_bar[gs], (uint32_t)((gq / ns) - 1) & 1u, abort_flag, p.wait_ns)))
              stop = 1;
            if (__any_sync(0xffffffffu, stop != 0)) {
              aborted = true;
              break;
            }
            if (in) {
              int32_t y = -2 * kPage;  // fully out of bounds: the TMA fills zeros
              if (page >= 0 && page < p.num_pages) y = (page * p.Hkv + hh) * kPage;
              else flag(p.dev_status, RGD_DEV_BAD_PAGE);
              descs[gs * kGroupPages + jpos] = (uint32_t)tok | ((uint32_t)(rowsel & 0xffff) << 16);
              uint8_t* sl = smem + gs * kSlot;
              mbar_arrive_expect_tx(&full_bar[gs], kStage);
              if (jpos == ng - 1 && ng < kGroupPages) mbar_arrive_cnt(&full_bar[gs], kGroupPages - ng);
#pragma unroll
              for (int hf = 0; hf < kHalves; ++hf)
                tma_load_3d_hint(sl + hf * (kGroupPages * 2048) + jpos * 2048, &tmK, &full_bar[gs], 0, y, hf, pol);
              tma_load_3d_hint(sl + kVOff + jpos * kTile, &tmV, &full_bar[gs], 0, y, 0, pol);
              if (start) {
                atomicMax(&s_issued, gq + 1);
                atomicMax(&s_slot_gen[gs], gq);
              }
            }
          }
          if (aborted) break;
        }
        gbase += __popc(starts);
      }
    }
    // Every copy of this block is issued: a programmatic dependent of this
    // kernel (the sample head) may be scheduled once every block has got here
    // or exited.  It still waits for this kernel to complete before it reads.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  } else if (warp == kMmaWarp) {
    // ============================ QK issue ============================
    // One thread issues S = Q K^T for every group as soon as its pages have
    // landed and its S / P buffer is free; the PV MMAs come from another warp,
    // since an issuing thread spends ~60 cycles per MMA whatever its size (two
    // issuers double the MMA rate; N = 64 MMAs take the tensor pipe ~32 cycles).
    // B descriptors are formed once; an MMA's B differs from the ring base only
    // in the start-address field (byte offset / 16).
    if (lane == 0 && b < e) {
      const uint64_t k_d = smem_desc(sbase, 1024, 1024, 2);
      int gi = 0, pc = 0;
      bool ok = true;
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      for (bool more = b < e; ok && more; more = next_piece(p, gpre, it, pc, cur, n_in)) {
        if (!wait_or_abort(&q_full, (uint32_t)pc & 1u, abort_flag, p.wait_ns)) break;
        tc_fence_after();
        const uint32_t qa = tmem + kQCol;
        for (int k0 = 0; k0 < n_in; k0 += kGroupPages) {
          const int ng = min(kGroupPages, n_in - k0);
          const int sb = gi % kSBufs;
          const int gs = gi % ns;
          if (!wait_or_abort(&full_bar[gs], (uint32_t)(gi / ns) & 1u, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          // the S buffer is free once the softmax has read the group that used it last
          if (gi >= kSBufs && !wait_or_abort(&s_empty[sb], (uint32_t)((gi / kSBufs) - 1) & 1u, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t idesc_qk = idesc_bf16_f32(kRows, kPage * ng, 0, 0);
          const uint64_t kg = k_d + (uint64_t)((gs * kSlot) >> 4);
          const uint32_t dcol = tmem + kSCol + sb * 64;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk)
            umma_bf16_tmem_a(dcol, qa + kk * 8,
                             kg + (uint64_t)(((kk >> 2) * (kGroupPages * 2048) + (kk & 3) * 32) >> 4), idesc_qk,
                             kk > 0 ? 1u : 0u);
          umma_commit(&s_full[sb]);
          if (k0 + ng == n_in) umma_commit(&q_empty);  // Q may take the next piece
          ++gi;
        }
        ++pc;
      }
    }
  } else if (warp == kPvWarp) {
    // ============================ PV issue ============================
    // O += P V for every page of a group once the softmax has written its P
    // (and, for a piece's first group, once the previous piece's O has been
    // read); one commit then frees the S / P buffer, another the ring slot.
    if (lane == 0 && b < e) {
      const uint64_t v_d = smem_desc(sbase, D == 128 ? kVLbo : 1024, D == 128 ? kVSbo : 1024, 2);
      int gi = 0, pc = 0;
      bool ok = true;
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      for (bool more = b < e; ok && more; more = next_piece(p, gpre, it, pc, cur, n_in)) {
        for (int k0 = 0; k0 < n_in; k0 += kGroupPages) {
          const int ng = min(kGroupPages, n_in - k0);
          const int pb = gi % kPBufs;
          const int gs = gi % ns;
          if (!wait_or_abort(&p_full[pb], (uint32_t)(gi / kPBufs) & 1u, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          // a piece's O buffer is free once the piece two back has been read out
          if (k0 == 0 && pc >= 2 && !wait_or_abort(&o_free[pc & 1], (uint32_t)((pc >> 1) - 1) & 1u, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // P = bf16 high part + bf16 residual: two MMAs per page keep ~16 bits of P
#pragma unroll
          for (int j = 0; j < kGroupPages; ++j) {
            if (j < ng) {
              const uint64_t vd = v_d + (uint64_t)((gs * kSlot + kVOff + j * kTile) >> 4);
              const uint32_t od = tmem + kOCol + (pc & 1) * kOStride;
              umma_bf16_tmem_a(od, tmem + kPCol + pb * 32 + j * 8, vd, kIdescPV, (k0 == 0 && j == 0) ? 0u : 1u);
              umma_bf16_tmem_a(od, tmem + kPLoCol + pb * 32 + j * 8, vd, kIdescPV, 1u);
            }
          }
          umma_commit(&p_empty[pb]);
          umma_commit(&empty_bar[gs]);  // the slot's K and V are no longer read
          if (k0 + ng == n_in) umma_commit(&o_full[pc & 1]);  // the piece's O is final
          ++gi;
        }
        ++pc;
      }
    }
  } else {
    // ============================ softmax / epilogue =================
    // The nq query rows span qpc = ceil(nq / 32) TMEM lane quarters, so R = 4 / qpc
    // copies of them fit in the 128 lanes (Q is written R times; S costs the
    // same MMAs either way).  Copy c handles pages c, c + R, ... of every group
    // with an online softmax of its own, and W = 4 / R warps of each of its
    // quarters (one page each) share that copy's running max; its P is zero in
    // the other copies' page columns, so O in its lanes sums its own pages only.
    // For nq <= 32 each page of a group is thus handled on its own SM
    // sub-partition (a warp can only reach its own lane quarter) and no warp
    // waits for another between groups.
    // The other 4 - W warps of each used quarter are the epilogue warps: they
    // write the next piece's Q and, while the softmax warps go on with the next
    // piece (into the other O buffer), read a finished piece's O, merge the
    // copies by log-sum-exp through shared memory and write the output or the
    // partial.  With W = 4 (no spare warps) the softmax warps do both in turn.
    const int nq = p.nq, gq = p.gq;
    const int qd = warp & 3, pj = warp >> 2;  // TMEM lane quarter; warp within the quarter
    const int cp = qd / qpc, rb = qd % qpc;   // copy; row block of the queries
    const bool in_piece = cp < R;
    const bool in_group = in_piece && pj < W;
    const bool in_epi = in_piece && (side ? pj >= W : true);
    const int ei = side ? pj - W : pj;        // index among the quarter's epilogue warps (< NE)
    const int jp = cp + pj * R;               // a softmax warp's page within a group
    auto soft_sync = [&]() { asm volatile("bar.sync 1, %0;" ::"r"(n_soft * 32) : "memory"); };
    auto epi_sync = [&]() { asm volatile("bar.sync 2, %0;" ::"r"(n_epi * 32) : "memory"); };
    const int r = rb * 32 + lane;              // this thread's query
    const int rloc = r < nq ? r / gq : -2;     // its row within the group (suffix pages are per row)
    const int tlane = qd * 32 + lane;          // its TMEM lane
    const uint32_t tl = tmem + ((uint32_t)(qd * 32) << 16);
    float* rmax = reinterpret_cast<float*>(smem + L.red);  // [2][4][128] page-slot maxima
    float* rsum = rmax + 2 * 4 * kRows;                    // [2 pieces][4][128] page-slot row sums
    float* mfin = rsum + 2 * 4 * kRows;                    // [2 pieces][128] running max at the piece end
    float4* stage = reinterpret_cast<float4*>(mfin + 2 * kRows);  // [2][<= 3][4][32] O columns of copies >= 1
    const int ocols = D / W;                   // O columns rescaled by each softmax warp of a quarter
    float* pref_o = reinterpret_cast<float*>(smem + L.pref);                        // [npref][nq][D + 4]
    float2* pref_ml = reinterpret_cast<float2*>(pref_o + p.npref * nq * (D + 4));   // [npref][ml_stride(nq)]
    int n_pref = 0;  // prefetches completed (the parity of pref_bar)
    constexpr int kChunks = D / 16;            // 16-column chunks of O (and 8-column chunks of Q)
    // warp-uniform bounded wait (TMEM loads and stores that follow are warp-collective)
    auto wwait = [&](uint64_t* bar, uint32_t parity, volatile int32_t* flag) {
      return __all_sync(0xffffffffu, wait_or_abort(bar, parity, flag, p.wait_ns));
    };
    // Q of job jb: this epilogue warp's share of its rows' query columns (8-column
    // chunks ei, ei + NE, ...), loaded first; then, if `after` is set, the wait for
    // the last QK of the piece before, which frees the single Q buffer
    // (the loads are issued before the wait for q_empty, which `waitf` does)
    auto write_q = [&](const Job& jb, bool after, uint32_t parity, auto&& waitf) {
      constexpr int kMaxChunks = (kChunks + NE - 1) / NE;
      uint4 qv[2 * kMaxChunks];
      int n = 0;
      const bool qrow = r < nq;
      const uint4* src = nullptr;
      if (qrow) {
        const int rr = jb.g * p.rpg + r / gq, hq = jb.h * gq + r % gq;
        src = reinterpret_cast<const uint4*>(p.q + ((int64_t)rr * p.Hq + hq) * D);
      }
#pragma unroll
      for (int t = 0; t < kMaxChunks; ++t) {
        const int ch = ei + t * NE;
        if (t * NE < kChunks && ch < kChunks) {
          qv[2 * t] = qrow ? __ldg(src + 2 * ch) : make_uint4(0u, 0u, 0u, 0u);
          qv[2 * t + 1] = qrow ? __ldg(src + 2 * ch + 1) : make_uint4(0u, 0u, 0u, 0u);
          n = t + 1;
        }
      }
      bool fine = true;
      if (after && !waitf(&q_empty, parity)) fine = false;
      if (fine) {
        tc_fence_after();
#pragma unroll
        for (int t = 0; t < kMaxChunks; ++t) {
          if (t < n) {
            const uint32_t v8[8] = {qv[2 * t].x,     qv[2 * t].y,     qv[2 * t].z,     qv[2 * t].w,
                                    qv[2 * t + 1].x, qv[2 * t + 1].y, qv[2 * t + 1].z, qv[2 * t + 1].w};
            tmem_st8(tl + kQCol + (ei + t * NE) * 8, v8);
          }
        }
        tmem_st_wait();
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&q_full);
      return fine;
    };

    // P columns of pages this warp's copy does not handle must read 0 in its
    // lanes: they are never written after this
    if (in_group) {
      const uint32_t zero[16] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
#pragma unroll
      for (int c0 = 0; c0 < 2 * kPBufs * 32; c0 += 16) tmem_st16(tl + kPCol + c0, zero);  // high and residual
      tmem_st_wait();
    }

    // jobs with no pages at all (empty prompt and suffixes, some row active)
    for (int j = c; j < p.G * p.Hkv; j += p.C) {
      const int g = j / p.Hkv, h = j % p.Hkv;
      if (gpre[g + 1] != gpre[g]) continue;
      for (int idx = tid; idx < nq * D; idx += kSoftThreads) {
        const int i = idx / D, d = idx % D;
        const int rr = g * p.rpg + i / gq, hq = h * gq + i % gq;
        if (!row_on(p, rr)) continue;
        p.out[((int64_t)rr * p.Hq + hq) * D + d] = __float2bfloat16(0.f);
        if (d == 0 && p.lse) p.lse[(int64_t)rr * p.Hq + hq] = -INFINITY;
      }
    }

    // These warps never leave their loops early: the loop structure is the same
    // for all warps of a role, so every named barrier is reached even after an
    // abort (waits then return at once and the work is skipped).
    int gi = 0;
    bool ok = true;
    // the groups of one job piece (softmax warps), then the hand-off of the
    // piece's (m, l) to the epilogue warps
    auto run_groups = [&](const Job& cur, int n_in, int pc) {
      const int ob = pc & 1;
      const uint32_t ocol = kOCol + ob * kOStride;
        float m_used = -INFINITY, l = 0.f;  // m_used is shared by the W warps of a quarter; l is per warp
        for (int k0 = 0; k0 < n_in; k0 += kGroupPages) {
          const int ng = min(kGroupPages, n_in - k0);
          const int sb = gi % kSBufs, pb = gi % kPBufs, gs = gi % ns;
          const bool has = jp < ng;
          int tok = 0, sel = -1;
          if (has && ok) {
            // this page's descriptor; the producer's write is ordered by the full barrier
            if (wwait(&full_bar[gs], (uint32_t)(gi / ns) & 1u, abort_flag)) {
              const uint32_t dsc = descs[gs * kGroupPages + jp];
              tok = (int)(dsc & 0xffffu);
              sel = (int)(int16_t)(dsc >> 16);
            } else {
              ok = false;
            }
          }
          if (ok && !wwait(&s_full[sb], (uint32_t)(gi / kSBufs) & 1u, abort_flag)) ok = false;
          tc_fence_after();
          float sc[kPage];
#pragma unroll
          for (int t = 0; t < kPage; ++t) sc[t] = -INFINITY;
          if (has && ok) {
            uint32_t raw[16];
            tmem_ld16(tl + kSCol + sb * 64 + jp * kPage, raw);
            tmem_ld_wait();
#pragma unroll
            for (int t = 0; t < kPage; ++t) sc[t] = __uint_as_float(raw[t]);
          }
          // S is in registers: its buffer can take the group after next
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s_empty[sb]);
          // masks: token count of the page, and a suffix page is visible to one row only
          const bool rowok = has && ok && rloc >= 0 && (sel < 0 || sel == rloc);
#pragma unroll
          for (int t = 0; t < kPage; ++t) sc[t] = (rowok && t < tok) ? sc[t] * p.scale_log2 : -INFINITY;
          float mx = fmaxf(fmaxf(fmaxf(fmaxf(sc[0], sc[1]), fmaxf(sc[2], sc[3])), fmaxf(fmaxf(sc[4], sc[5]), fmaxf(sc[6], sc[7]))),
                           fmaxf(fmaxf(fmaxf(sc[8], sc[9]), fmaxf(sc[10], sc[11])), fmaxf(fmaxf(sc[12], sc[13]), fmaxf(sc[14], sc[15]))));
          if (W > 1) {
            // the group's row max over the quarter's page slots
            float* rm = rmax + (gi & 1) * 4 * kRows;
            rm[pj * kRows + tlane] = mx;
            soft_sync();
            mx = rm[tlane];
            for (int w = 1; w < W; ++w) mx = fmaxf(mx, rm[w * kRows + tlane]);
          }
          const bool need = mx > m_used + kRescaleLog2;
          if (__any_sync(0xffffffffu, need)) {
            const float nm = need ? mx : m_used;
            const float f = (m_used == -INFINITY) ? 0.f : exp2f(m_used - nm);
            const int pg = gi - 1;
            if (k0 > 0 && ok && !wwait(&p_empty[pg % kPBufs], (uint32_t)(pg / kPBufs) & 1u, abort_flag)) ok = false;
            if (k0 > 0 && ok) {
              // O holds this piece's earlier groups: the last PV is done; rescale this warp's columns
              tc_fence_after();
#pragma unroll 1
              for (int cc = 0; cc < ocols; cc += 16) {
                uint32_t raw[16];
                const uint32_t col = ocol + pj * ocols + cc;
                tmem_ld16(tl + col, raw);
                tmem_ld_wait();
#pragma unroll
                for (int t = 0; t < 16; ++t) raw[t] = __float_as_uint(__uint_as_float(raw[t]) * f);
                tmem_st16(tl + col, raw);
              }
              tmem_st_wait();
            }
            l *= f;
            m_used = nm;
          }
          // P = 2^(s - m) (ex2 of -inf is +0: masked tokens give 0)
          const float ref = (m_used == -INFINITY) ? 0.f : m_used;
          float pv[kPage];
#pragma unroll
          for (int t = 0; t < kPage; ++t) pv[t] = ex2_approx(sc[t] - ref);
          // P in bf16 as a high part and the residual (P - high), each bf16
          uint32_t pk[kPage / 2], pl[kPage / 2];
#pragma unroll
          for (int t = 0; t < kPage; t += 2) {
            pk[t / 2] = pack_bf16x2(pv[t], pv[t + 1]);
            const float h0 = __uint_as_float(pk[t / 2] << 16), h1 = __uint_as_float(pk[t / 2] & 0xffff0000u);
            pl[t / 2] = pack_bf16x2(pv[t] - h0, pv[t + 1] - h1);
          }
          l += ((((pv[0] + pv[1]) + (pv[2] + pv[3])) + ((pv[4] + pv[5]) + (pv[6] + pv[7]))) +
                (((pv[8] + pv[9]) + (pv[10] + pv[11])) + ((pv[12] + pv[13]) + (pv[14] + pv[15]))));
          // the P buffer is free once the PV of the group that used it last is done
          const int pq = gi - kPBufs;
          if (pq >= 0 && ok && !wwait(&p_empty[pb], (uint32_t)(pq / kPBufs) & 1u, abort_flag)) ok = false;
          if (has && ok) {
            tc_fence_after();
            tmem_st8(tl + kPCol + pb * 32 + jp * 8, pk);  // P of this page (the other copies' pages stay 0)
            tmem_st8(tl + kPLoCol + pb * 32 + jp * 8, pl);
            tmem_st_wait();
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&p_full[pb]);
          ++gi;
        }
        // hand the piece's (m, l) to the epilogue warps (slot reused two pieces on)
        if (pc >= 2 && ok && !wwait(&ml_empty[ob], (uint32_t)((pc >> 1) - 1) & 1u, abort_flag)) ok = false;
        rsum[(ob * 4 + pj) * kRows + tlane] = l;
        if (pj == 0) mfin[ob * kRows + tlane] = m_used;
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_full[ob]);
          };
    // Merge of a split job's partials by the epilogue threads, one piece at a
    // time: bulk copies bring the piece's partial into the prefetch area and
    // each thread folds it into its items (item = 4 output columns of one
    // query), kU items at a time: with piece s holding the unnormalised o_s and
    // (m_s, l_s) in log2 units, out = sum 2^(m_s - M) o_s / sum 2^(m_s - M) l_s.
    auto merge_staged = [&](const Job& jb, int jj, int first, int last, int et, int n_et) {
      merge_from_l2<D>(p.slot_ml, p.slot_o, p.out, p.lse, nq, gq, p.rpg, p.Hq, jb.g, jb.h, jj, first, last, et, n_et,
                       rowbits, !*abort_flag);
    };
    // the next piece's Q, then this piece's end (epilogue warps)
    auto run_epilogue = [&](const Job& cur, int pc, bool more, const Job& nxt) {
      const int j = cur.g * p.Hkv + cur.h;
      const int ob = pc & 1;
      const uint32_t ocol = kOCol + ob * kOStride;
      const int first = cta_of(cur.start, T, Ceff), last = cta_of(cur.start + cur.n - 1, T, Ceff);
      const int rr = r < nq ? cur.g * p.rpg + r / gq : 0, hq = r < nq ? cur.h * gq + r % gq : 0;
      const bool mine_row = r < nq && cp == 0;
      const bool write_row = mine_row && ((rowbits[rr >> 5] >> (rr & 31)) & 1u);
      const int et = (ei * (R * qpc) + qd) * 32 + lane;  // index among the epilogue threads
      const int n_et = n_epi * 32;
      const bool watcher = ei == 0 && qd == 0;           // the warp holding et == 0
      // A split job is merged by the block holding its first page (the merger);
      // its other pieces (each the first piece of its own block, so never
      // behind a wait on another block) write a partial and count themselves
      // in the job's ticket (an aborted piece also in the high half).  The
      // merger's watcher warp watches the ticket while this piece runs and,
      // once the count is complete, has bulk copies bring the partials into
      // shared memory; the merger then folds them into its own O on the way out.
      const bool split = first != last;
      const int nparts = last - first;  // the job's other pieces
      const bool merger = split && c == first;
      const bool staged = merger && nparts <= p.npref;  // the partials fit the prefetch area
      auto issue_prefetch = [&]() {                       // (the watcher warp, all lanes)
        const int mls = ml_stride(nq);
        if (lane == 0) {
          mbar_arrive_expect_tx(&pref_bar, (uint32_t)(nparts * (nq * D * 4 + mls * 8)));
          ++s_pref_n;
        }
        __syncwarp();
        fence_proxy_async_global();  // the partials were seen by the generic proxy (the acquire)
        for (int it = lane; it < nparts * (nq + 1); it += 32) {
          const int k = it / (nq + 1), i = it % (nq + 1);
          const int64_t sl = (int64_t)(first + k + 1) + j;  // the k-th other piece's slot
          if (i < nq) bulk_load(pref_o + (k * nq + i) * (D + 4), p.slot_o + (sl * nq + i) * D, D * 4, &pref_bar);
          else bulk_load(pref_ml + k * mls, p.slot_ml + sl * mls, mls * 8, &pref_bar);
        }
      };
      // (watcher) the ticket once its count is complete (0: not seen yet), and
      // whether the partner copies are on their way
      int tk = 0;
      bool issued = false;
      const bool polling = staged && watcher;
      // the ticket read is consumed a few sleeps later, so that a wait never
      // stalls on it once its barrier has completed
      int pend = polling && lane == 0 ? ld_acquire_gpu(p.ticket + j) : 0;
      auto seen = [&](int t) {
        if ((t & 0xffff) != nparts) return false;
        tk = t;
        if (staged && (t >> 16) == 0 && __all_sync(0xffffffffu, ok)) {  // (only staged partials fit the area)
          issue_prefetch();
          issued = true;
        }
        return true;
      };
      // A bounded wait on `bar`, during which the watcher polls the ticket.
      auto wait_polling = [&](uint64_t* bar, uint32_t par) -> bool {
        if (!polling || !__all_sync(0xffffffffu, ok)) return ok && wwait(bar, par, abort_flag);
        // (a non-blocking test and short sleeps: a blocking try_wait would
        // return only once the phase completes)
        const uint64_t t0 = globaltimer_ns();
        for (uint32_t i = 1;; ++i) {
          if (__any_sync(0xffffffffu, mbar_test_wait(bar, par))) return true;
          if (tk == 0 && (i & 7u) == 0 && !seen(__shfl_sync(0xffffffffu, pend, 0)) && lane == 0)
            pend = ld_acquire_gpu(p.ticket + j);
          __nanosleep(200);
          if ((i & 63u) == 0) {  // (warp-uniform exits: the loop holds warp collectives)
            if (__any_sync(0xffffffffu, *abort_flag != 0)) return false;
            if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > p.wait_ns)) {
              *abort_flag = 1;
              return false;
            }
          }
        }
      };
      // (watcher) Bounded wait until the job's other pieces have all counted
      // themselves: they never wait on this block, so it ends; it is also
      // waited for after an abort, so that the merger can clear the ticket.
      auto wait_ticket = [&]() {
        const uint64_t t0 = globaltimer_ns();
        while (tk == 0) {
          if (seen(__shfl_sync(0xffffffffu, lane == 0 ? ld_acquire_gpu(p.ticket + j) : 0, 0))) break;
          if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > p.wait_ns)) {
            *abort_flag = 1;
            tk = -1;
            break;
          }
          __nanosleep(256);
        }
      };
      // ---- the next piece's Q, once this piece's last QK is done ----
      if (more && !write_q(nxt, true, (uint32_t)pc & 1u, wait_polling)) ok = false;
      // ---- this piece's epilogue: O is final once its last PV completes ----
      if (!wait_polling(&o_full[ob], (uint32_t)(pc >> 1) & 1u)) ok = false;
      if (ok && !wwait(&ml_full[ob], (uint32_t)(pc >> 1) & 1u, abort_flag)) ok = false;
      tc_fence_after();
      // the copies' running maxima and row sums -> the piece's max M and sum L;
      // copy c's O is weighted by 2^(m_c - M)
      float M = -INFINITY, Ls = 0.f;
      for (int c2 = 0; c2 < R; ++c2) M = fmaxf(M, mfin[ob * kRows + (c2 * qpc + rb) * 32 + lane]);
      for (int c2 = 0; c2 < R; ++c2) {
        const int ln = (c2 * qpc + rb) * 32 + lane;
        float Lc = 0.f;
        for (int w = 0; w < W; ++w) Lc += rsum[(ob * 4 + w) * kRows + ln];
        const float mc = mfin[ob * kRows + ln];
        if (mc != -INFINITY) Ls += exp2f(mc - M) * Lc;
      }
      const float mself = mfin[ob * kRows + tlane];
      const float wself = mself == -INFINITY ? 0.f : exp2f(mself - M);
      __syncwarp();
      if (lane == 0) mbar_arrive(&ml_empty[ob]);  // the (m, l) slot has been read
      const int64_t s_idx = (int64_t)c + j;
      // fused: a merger whose partners' partials are (being) staged folds them
      // in here, with its own O still in registers
      bool fused = false, partners_ok = true;
      if (staged) {
        if (watcher) {
          wait_ticket();
          if (lane == 0) s_last = issued ? 1 : 0;  // 0: a piece (or this block) gave up
        }
        epi_sync();
        fused = true;
        partners_ok = s_last == 1;
        if (partners_ok) {
          if (!wwait(&pref_bar, (uint32_t)n_pref & 1u, abort_flag)) ok = false;  // the partials have landed
          ++n_pref;
        }
      }
      // after an abort the piece's outputs are not written (the status word says so)
      const bool out_ok = __all_sync(0xffffffffu, ok && !*abort_flag) && partners_ok;
      // this piece's weight a and the partners' b_k in the merged softmax:
      // out = (a o + sum_k b_k o_k) / (a L + sum_k b_k l_k)
      float Mt = M, Lt = Ls, a = 1.f, bk[2] = {0.f, 0.f};
      if (fused && out_ok && r < nq) {
        Mt = Ls > 0.f ? M : -INFINITY;
        float2 ml[2];
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          ml[k] = k < nparts ? pref_ml[k * ml_stride(nq) + r] : make_float2(-INFINITY, 0.f);
          if (ml[k].y > 0.f) Mt = fmaxf(Mt, ml[k].x);
        }
        a = Ls > 0.f ? exp2f(M - Mt) : 0.f;
        Lt = a * Ls;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          bk[k] = ml[k].y > 0.f ? exp2f(ml[k].x - Mt) : 0.f;
          Lt += bk[k] * ml[k].y;
        }
      }
      const float inv = Lt > 0.f ? 1.f / Lt : 0.f;
      // The block's last piece, with copies: the ring is idle (every group's
      // PV is done), so it holds all the copies' O at once -- each epilogue
      // warp writes its copy's columns there, one barrier, and the R warps of a
      // row block then each sum the copies over their own D/R columns and
      // write those (instead of one barrier per 16 columns and copy 0's warp
      // writing every column).
      const bool whole = R > 1 && !more;
      if (whole) {
        float* stg = reinterpret_cast<float*>(smem);  // [R * qpc][D][32]
        float* mine = stg + (size_t)(cp * qpc + rb) * D * 32;
        if (out_ok) {
#pragma unroll 1
          for (int col = 0; col < D; col += 32) {
            uint32_t r0[16], r1[16];
            tmem_ld16(tl + ocol + col, r0);
            tmem_ld16(tl + ocol + col + 16, r1);
            tmem_ld_wait();
#pragma unroll
            for (int t = 0; t < 16; ++t) {
              mine[(col + t) * 32 + lane] = __uint_as_float(r0[t]) * wself;
              mine[(col + 16 + t) * 32 + lane] = __uint_as_float(r1[t]) * wself;
            }
          }
        }
        epi_sync();
        constexpr int kCols = D / R;  // this warp's output columns (a multiple of 16)
        const bool row_ok = out_ok && r < nq;
        const bool out_row = row_ok && ((rowbits[rr >> 5] >> (rr & 31)) & 1u);
#pragma unroll 1
        for (int c0 = 0; c0 < kCols; c0 += 16) {
          const int col = cp * kCols + c0;
          if (!row_ok) break;
          float o[16];
#pragma unroll
          for (int t = 0; t < 16; ++t) o[t] = 0.f;
          for (int c2 = 0; c2 < R; ++c2) {
            const float* src = stg + ((size_t)(c2 * qpc + rb) * D + col) * 32 + lane;
#pragma unroll
            for (int t = 0; t < 16; ++t) o[t] += src[t * 32];
          }
          if (!split || fused) {
            if (!out_row) continue;
            if (fused) {
#pragma unroll
              for (int t = 0; t < 16; ++t) o[t] *= a;
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                if (k >= nparts) break;
                const float4* src4 = reinterpret_cast<const float4*>(pref_o + (k * nq + r) * (D + 4) + col);
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                  const float4 v = src4[t];
                  o[4 * t] += bk[k] * v.x;
                  o[4 * t + 1] += bk[k] * v.y;
                  o[4 * t + 2] += bk[k] * v.z;
                  o[4 * t + 3] += bk[k] * v.w;
                }
              }
            }
            uint4* dst = reinterpret_cast<uint4*>(p.out + ((int64_t)rr * p.Hq + hq) * D + col);
            dst[0] = make_uint4(pack_bf16x2(o[0] * inv, o[1] * inv), pack_bf16x2(o[2] * inv, o[3] * inv),
                                pack_bf16x2(o[4] * inv, o[5] * inv), pack_bf16x2(o[6] * inv, o[7] * inv));
            dst[1] = make_uint4(pack_bf16x2(o[8] * inv, o[9] * inv), pack_bf16x2(o[10] * inv, o[11] * inv),
                                pack_bf16x2(o[12] * inv, o[13] * inv), pack_bf16x2(o[14] * inv, o[15] * inv));
          } else {
            float4* dst = reinterpret_cast<float4*>(p.slot_o + (s_idx * nq + r) * D + col);
#pragma unroll
            for (int t = 0; t < 4; ++t) dst[t] = make_float4(o[4 * t], o[4 * t + 1], o[4 * t + 2], o[4 * t + 3]);
          }
        }
      }
      // Otherwise O in 16-column chunks: epilogue warp ei of a quarter takes
      // chunks ei, ei + NE, ...; copies >= 1 pass theirs to copy 0 through
      // shared memory
      constexpr int rounds = (kChunks + NE - 1) / NE;
      const int my_stage = ((cp - 1) * qpc + rb) * NE + ei;  // (for copies >= 1)
#pragma unroll 1
      for (int rd = 0; rd < (whole ? 0 : rounds); ++rd) {
        const int ch = ei + rd * NE;
        const bool has = ch < kChunks && out_ok;
        const int col = ch * 16;
        float o[16];
        if (has) {
          uint32_t raw[16];
          tmem_ld16(tl + ocol + col, raw);
          tmem_ld_wait();
#pragma unroll
          for (int t = 0; t < 16; ++t) o[t] = __uint_as_float(raw[t]) * wself;
        }
        if (R > 1) {
          // double-buffered: a round's staging is rewritten two rounds later,
          // after the next round's barrier, which copy 0 passes only once it
          // has read it
          float4* stg = stage + (rd & 1) * (3 * 4 * 32);
          if (cp > 0 && has) {
#pragma unroll
            for (int t = 0; t < 4; ++t)
              stg[(my_stage * 4 + t) * 32 + lane] = make_float4(o[4 * t], o[4 * t + 1], o[4 * t + 2], o[4 * t + 3]);
          }
          epi_sync();
          if (cp == 0 && has) {
#pragma unroll
            for (int c2 = 1; c2 < R; ++c2) {
              const float4* src4 = stg + ((((c2 - 1) * qpc + rb) * NE + ei) * 4) * 32 + lane;
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                const float4 v = src4[t * 32];
                o[4 * t] += v.x;
                o[4 * t + 1] += v.y;
                o[4 * t + 2] += v.z;
                o[4 * t + 3] += v.w;
              }
            }
          }
        }
        if (!has) continue;
        if (!split || fused) {
          if (write_row) {
            if (fused) {
#pragma unroll
              for (int t = 0; t < 16; ++t) o[t] *= a;
#pragma unroll
              for (int k = 0; k < 2; ++k) {
                if (k >= nparts) break;
                const float4* src4 = reinterpret_cast<const float4*>(pref_o + (k * nq + r) * (D + 4) + col);
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                  const float4 v = src4[t];
                  o[4 * t] += bk[k] * v.x;
                  o[4 * t + 1] += bk[k] * v.y;
                  o[4 * t + 2] += bk[k] * v.z;
                  o[4 * t + 3] += bk[k] * v.w;
                }
              }
            }
            uint4* dst = reinterpret_cast<uint4*>(p.out + ((int64_t)rr * p.Hq + hq) * D + col);
            dst[0] = make_uint4(pack_bf16x2(o[0] * inv, o[1] * inv), pack_bf16x2(o[2] * inv, o[3] * inv),
                                pack_bf16x2(o[4] * inv, o[5] * inv), pack_bf16x2(o[6] * inv, o[7] * inv));
            dst[1] = make_uint4(pack_bf16x2(o[8] * inv, o[9] * inv), pack_bf16x2(o[10] * inv, o[11] * inv),
                                pack_bf16x2(o[12] * inv, o[13] * inv), pack_bf16x2(o[14] * inv, o[15] * inv));
          }
        } else if (mine_row) {
          float4* dst = reinterpret_cast<float4*>(p.slot_o + (s_idx * nq + r) * D + col);
#pragma unroll
          for (int t = 0; t < 4; ++t) dst[t] = make_float4(o[4 * t], o[4 * t + 1], o[4 * t + 2], o[4 * t + 3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free[ob]);  // this O buffer may take the piece after next
      if (!split || fused) {
        if (out_ok && ei == 0 && write_row && p.lse)
          p.lse[(int64_t)rr * p.Hq + hq] = Lt > 0.f ? (Mt + log2f(Lt)) * kLn2 : -INFINITY;
        if (fused && et == 0) p.ticket[j] = 0;  // every other piece has counted itself
        if (R > 1 || fused) epi_sync();         // staging and prefetch areas are reused at the next piece
        return;
      }
      // this piece's partial, visible before its count
      if (out_ok && ei == 0 && mine_row) p.slot_ml[s_idx * ml_stride(nq) + r] = make_float2(M, Ls);
      __threadfence();
      epi_sync();
      if (!merger) {
        if (et == 0) atomicAdd(p.ticket + j, out_ok && !*abort_flag ? 1 : 0x10001);
        return;
      }
      // a merger whose partners' partials do not fit the prefetch area: once
      // they have all counted themselves, merge every piece's partial
      if (watcher) {
        wait_ticket();
        if (lane == 0) s_last = tk > 0 && (tk >> 16) == 0 && !*abort_flag ? 1 : 0;
      }
      epi_sync();
      if (s_last == 1) {
        __threadfence();
        merge_staged(cur, j, first, last, et, n_et);
      }
      if (et == 0) p.ticket[j] = 0;
      epi_sync();  // (the prefetch area and s_last are reused at the next piece)
    };
    if (in_piece && b < e) {
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      if (in_epi && !write_q(cur, false, 0u, [](uint64_t*, uint32_t) { return true; })) ok = false;
      for (int pc = 0;; ++pc) {
        Job nxt = cur;
        int n_nxt = n_in;
        const bool more = next_piece(p, gpre, it, pc + 1, nxt, n_nxt);
        if (side) {
          // one role per warp: the softmax warps run ahead into the next piece
          // while the epilogue warps finish this one
          if (in_group) run_groups(cur, n_in, pc);
          else run_epilogue(cur, pc, more, nxt);
        } else {
          run_groups(cur, n_in, pc);
          run_epilogue(cur, pc, more, nxt);
        }
        if (!more) break;
        cur = nxt;
        n_in = n_nxt;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // a wait gave up: report, and let copies and MMAs still in flight drain (bounded)
    if (tid == 0) {
      flag(p.dev_status, RGD_DEV_WAIT_TIMEOUT);
      const int issued = s_issued;
      for (int g = max(0, issued - ns); g < issued; ++g) mbar_wait(&full_bar[g % ns], (g / ns) & 1);
      if (s_pref_n > 0) mbar_wait(&pref_bar, (uint32_t)(s_pref_n - 1) & 1u);  // the last partner prefetch
    }
    if ((warp == kMmaWarp || warp == kPvWarp) && lane == 0) {
      uint64_t* md = &mma_done[warp - kMmaWarp];
      umma_commit(md);  // arrives once every MMA this thread issued has completed
      mbar_wait(md, 0);
    }
    __syncthreads();
  }
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, kTmemCols);
}

}  // namespace
}  // namespace rgd

#include "attention_t.cuh"

namespace rgd {
namespace {

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

int make_kv_map(CUtensorMap* map, const void* base, int64_t rows, int D, int box_halves) {
  auto fn = get_encode_fn();
  if (!fn) return set_error(RGD_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  // View each 16-token page-head tile as (64 columns) x (16 rows) x (D/64 halves):
  // a box is one half or the whole tile, laid out in shared memory half-major
  // with the 128-byte swizzle (16-byte chunk index XOR row index mod 8).
  cuuint64_t dims[3] = {64, (cuuint64_t)rows, (cuuint64_t)(D / 64)};
  cuuint64_t strides[2] = {(cuuint64_t)D * 2, 128};
  cuuint32_t box[3] = {64, (cuuint32_t)kPage, (cuuint32_t)box_halves};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_error(RGD_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return RGD_OK;
}

// Limit of the kernel's waits on other roles and blocks, for the calls that
// follow (rgd_set_wait_limit_ns).
std::atomic<uint64_t> g_wait_ns{kWaitLimitNs};

int device_sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

struct Plan {
  int nq, nslots, C, J, npref;
  bool transposed;  // attn_t_kernel (nq <= 32) rather than attn_tc_kernel
  int smem_bytes;   // dynamic shared memory of the launch
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
  RGD_CHECK_ARG(s->num_ctas >= 0 && s->num_ctas <= 65535 && s->reserved == 0,
                "num_ctas must be in [0, 65535] and reserved 0");
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
  pl->C = s->num_ctas > 0 ? s->num_ctas : device_sm_count();
  if (pl->C <= 0) return set_error(RGD_ERR_CUDA, "could not query the device's SM count");
  pl->J = s->num_groups * s->num_kv_heads;
  // The ring holds at least three page groups: a group's slot is released by
  // its PV, which is issued after the next group's QK.
  // The shared memory holds the ring and, for the merge of a split job, one
  // or two partner partials (a job spans at most three blocks when blocks hold
  // about as many pages as a job).  Staging both partials is worth a ring slot
  // (it keeps the merges of three-piece jobs off the end of the blocks), down
  // to four slots; one staged partial is the minimum (the merges go through
  // that area).
  const int rows = s->num_groups * s->rows_per_group;
  pl->transposed = pl->nq <= kTN;
  pl->nslots = 0;
  pl->npref = 0;
  if (pl->transposed) {
    // as many 8-page group slots as fit (three at head dim 128, six at 64), at least two
    for (int ns = s->head_dim == 128 ? 3 : kTMaxSlots; ns >= 2; --ns) {
      const int tot = s->head_dim == 128 ? t_layout<128>(ns, s->num_groups, rows).total
                                         : t_layout<64>(ns, s->num_groups, rows).total;
      if (tot <= kSmemLimit) {
        pl->nslots = ns;
        pl->smem_bytes = tot;
        break;
      }
    }
    if (pl->nslots == 0)
      return set_error(RGD_ERR_UNSUPPORTED, "shape needs more shared memory than an SM has (too many groups?)");
  }
  auto layout = [&](int nslots, int npref) {
    return s->head_dim == 128 ? smem_layout<128>(nslots, s->num_groups, rows, pl->nq, npref)
                              : smem_layout<64>(nslots, s->num_groups, rows, pl->nq, npref);
  };
  for (int npref = 2; npref >= 1 && pl->nslots == 0; --npref) {
    for (int ns = kMaxSlots; ns >= (npref > 1 ? 4 : 3); --ns) {
      if (layout(ns, npref).total <= kSmemLimit) {
        pl->nslots = ns;
        pl->npref = npref;
        break;
      }
    }
  }
  if (pl->nslots == 0)
    return set_error(RGD_ERR_UNSUPPORTED, "shape needs more shared memory than an SM has (too many groups?)");
  if (!pl->transposed) pl->smem_bytes = layout(pl->nslots, pl->npref).total;
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  const size_t n_part = (size_t)pl->C + pl->J - 1;  // partial-result slots
  // The job counters come first, in an area of at least kTicketSlots counters
  // whatever the shape, so that a workspace reused for another shape with up to
  // kTicketSlots jobs finds its counters where earlier calls left zeros, not
  // where they wrote partials.
  pl->ticket_off = 0;
  pl->ml_off = up((size_t)std::max(pl->J, kTicketSlots) * sizeof(int32_t));
  pl->o_off = pl->ml_off + up(n_part * ml_stride(pl->nq) * sizeof(float2));
  pl->total = pl->o_off + up(n_part * pl->nq * s->head_dim * sizeof(float));
  return RGD_OK;
}

// Workspace fields used by the allocation-free entry point below.
size_t ws_total(const rgd_attn_shape* s) {
  Plan pl;
  return make_plan(s, &pl) == RGD_OK ? pl.total : 0;
}

}  // namespace
}  // namespace rgd

using namespace rgd;

extern "C" int rgd_set_wait_limit_ns(uint64_t limit_ns) {
  clear_error();
  g_wait_ns.store(limit_ns == 0 ? kWaitLimitNs : limit_ns, std::memory_order_relaxed);
  return RGD_OK;
}

extern "C" size_t rgd_prefix_decode_attn_workspace_size(const rgd_attn_shape* shape) {
  clear_error();
  Plan pl;
  if (make_plan(shape, &pl) != RGD_OK) return 0;
  return pl.total;
}

namespace rgd {
namespace {

// The attention kernel for one (head dim, copy count).
template <int D, int R>
int launch_attn(const CUtensorMap& tmK, const CUtensorMap& tmV, const AttnParams& p, const Plan& pl,
                cudaStream_t st) {
  static bool done = false;
  if (int rc = ensure_smem(attn_tc_kernel<D, R>, kSmemLimit, &done)) return rc;
  attn_tc_kernel<D, R><<<pl.C, Roles<R>::kThreads, pl.smem_bytes, st>>>(tmK, tmV, p);
  if (cudaError_t e = cudaGetLastError(); e != cudaSuccess) return cuda_error(e, "attention launch");
  return RGD_OK;
}

// The transposed attention kernel (jobs of at most 32 queries) for one head
// dim and NS softmax sets of 8 queries.
template <int D, int NS>
int launch_attn_t_ns(const CUtensorMap& tmK, const CUtensorMap& tmV, const AttnParams& p, const Plan& pl,
                     cudaStream_t st) {
  static bool done = false;
  if (int rc = ensure_smem(attn_t_kernel<D, NS>, kSmemLimit, &done)) return rc;
  attn_t_kernel<D, NS><<<pl.C, t_threads<NS>(), pl.smem_bytes, st>>>(tmK, tmV, p);
  if (cudaError_t e = cudaGetLastError(); e != cudaSuccess) return cuda_error(e, "attention launch");
  return RGD_OK;
}
template <int D>
int launch_attn_t(const CUtensorMap& tmK, const CUtensorMap& tmV, const AttnParams& p, const Plan& pl,
                  cudaStream_t st) {
  switch ((pl.nq + kTQS - 1) / kTQS) {  // softmax sets: one per 8 queries of a job
    case 1: return launch_attn_t_ns<D, 1>(tmK, tmV, p, pl, st);
    case 2: return launch_attn_t_ns<D, 2>(tmK, tmV, p, pl, st);
    case 3: return launch_attn_t_ns<D, 3>(tmK, tmV, p, pl, st);
    default: return launch_attn_t_ns<D, 4>(tmK, tmV, p, pl, st);
  }
}

}  // namespace
}  // namespace rgd

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
  if (int rc = make_kv_map(&tmK, k_pages, kv_rows, s.head_dim, 1)) return rc;                // one half per box
  if (int rc = make_kv_map(&tmV, v_pages, kv_rows, s.head_dim, s.head_dim / 64)) return rc;  // whole tile

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
  p.nslots = pl.nslots;
  p.npref = pl.npref;
  p.C = pl.C;
  p.scale_log2 = softmax_scale * kLog2e;
  p.wait_ns = g_wait_ns.load(std::memory_order_relaxed);

  cudaStream_t st = (cudaStream_t)stream;
  const int qpc = (pl.nq + 31) / 32;
  const int R = qpc == 1 ? 4 : qpc == 2 ? 2 : 1;  // copies of the queries in the TMEM lanes
  int rc = RGD_OK;
  if (pl.transposed) {
    rc = s.head_dim == 128 ? launch_attn_t<128>(tmK, tmV, p, pl, st) : launch_attn_t<64>(tmK, tmV, p, pl, st);
  } else if (s.head_dim == 128) {
    rc = R == 4 ? launch_attn<128, 4>(tmK, tmV, p, pl, st)
       : R == 2 ? launch_attn<128, 2>(tmK, tmV, p, pl, st)
                : launch_attn<128, 1>(tmK, tmV, p, pl, st);
  } else {
    rc = R == 4 ? launch_attn<64, 4>(tmK, tmV, p, pl, st)
       : R == 2 ? launch_attn<64, 2>(tmK, tmV, p, pl, st)
                : launch_attn<64, 1>(tmK, tmV, p, pl, st);
  }
  if (rc) return rc;
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? RGD_OK : cuda_error(e, "attention launch");
}

// ---------------------------------------------------------------------------
// Allocation-free variant of rgd_prefix_decode_attn
// ---------------------------------------------------------------------------
// The split partials live in a fixed file-scope device array
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
  // The counters must sit in the fixed area at the start of the array for every
  // shape (a larger job count would move the partials over them).
  if ((int64_t)shape->num_groups * shape->num_kv_heads > kTicketSlots)
    return set_error(RGD_ERR_UNSUPPORTED,
                     "rgd_prefix_decode_attn_noalloc: num_groups * num_kv_heads = %lld exceeds %d",
                     (long long)shape->num_groups * shape->num_kv_heads, kTicketSlots);
  const size_t need = ws_total(shape);
  if (need > kStaticScratchBytes)
    return set_error(RGD_ERR_UNSUPPORTED,
                     "rgd_prefix_decode_attn_noalloc: this shape needs %zu bytes of scratch; the static "
                     "scratch holds %zu (use rgd_prefix_decode_attn with a workspace)",
                     need, kStaticScratchBytes);
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
  // the array is zero when the module is loaded (device variables without an
  // initializer are zero-filled); every call leaves the counters of its jobs at
  // zero, and no call writes anything else into the fixed counter area
  return rgd_prefix_decode_attn(shape, q, k_pages, v_pages, prompt_block_table, prompt_len, suffix_block_table,
                                suffix_len, row_active, softmax_scale, out, lse, scratch, kStaticScratchBytes,
                                dev_status, stream);
}
