// Shared-prefix decode attention, transposed form, for jobs of at most 32
// queries (rows_per_group * Hq/Hkv <= 32: the Llama-3-8B-shaped, high-batch and
// tiny steps).  Included by attention.cu: same jobs, page order, block ranges,
// piece order, split-job merge protocol and workspace as attn_tc_kernel.
//
// With few queries per kv head, putting the queries on the MMA's M side (128
// rows) leaves most of every MMA idle.  Here the tokens are M and the queries
// are N:
//   S^T = K Q^T      A = a group's K (128 tokens = 8 pages, K-major), B = Q
//                    (32 query rows, K-major), accumulator S^T in 32 TMEM
//                    columns with token t in lane t;
//   O^T += V^T P^T   A = V^T of one page from TMEM (head dimension d in lane
//                    d, tokens along the columns), B = P^T of that page (16
//                    tokens x 32 queries, MN-major, in shared memory),
//                    accumulator O^T in 32 TMEM columns with d in lane d.
// So the tensor cores do no work for query copies, and a softmax thread owns
// one token: it reads that token's scores from its lane, and the query maxima
// are shared through shared memory only when one of them has to move (the
// reference maximum of a query is moved lazily, when a score exceeds it by more
// than 2^8; the first group of a piece always sets it).  P^T is written by the
// softmax threads as a bf16 high part and a bf16 residual into the group's K
// area, which its QK no longer needs, and each page's PV is two MMAs.  V lands
// token-major (as it is stored); the softmax threads copy it into TMEM with
// the head dimension in the lanes while the group's QK runs, because an A
// operand read from shared memory in MN-major order costs the tensor core
// twice the cycles of one read from TMEM.
//
// Warps: NS = ceil(nq / 8) softmax sets of four warps, set 0 at warps 0-3 and
// set s > 0 at warps 12 + 4(s - 1) .. +3 (lane quarter w & 3: tokens and, for
// the V^T copy, head dimensions 32(w & 3)..+31; set s takes queries 8s..8s+7
// and copies V^T of the group's pages s, s + NS, ...), 4-7 piece ends (lane
// quarter w - 4: head dimensions of O^T; they also write Q), 8 page producer,
// 9 PV issue of the P residuals, 10 QK issue (and the TMEM allocation), 11 PV
// issue of the P high parts.  Query columns past 8 NS are never used.
// TMEM: S^T x 2 (columns 0-63), O^T of the high parts x 2 by piece (64-127),
// V^T x 2 (128-255), O^T of the residuals x 2 by piece (256-319); the two O^T
// accumulate in parallel from two issuing threads and are summed at the piece
// end.

namespace rgd {
namespace {

constexpr int kTPages = 8;                  // pages per group: 128 tokens, the MMA's M
constexpr int kTN = 32;                     // query columns (the MMA's N); jobs with nq <= 32
constexpr int kTMaxSlots = 6;
constexpr int kTQS = 8;                     // queries per softmax set
template <int NS>
__host__ __device__ constexpr int t_threads() { return (4 * NS + 8) * 32; }
constexpr int kTEpi = 4, kTProd = 8, kTPvLo = 9, kTQk = 10, kTPv = 11, kTSoftB = 12;  // first warp of each role
constexpr int kTTmemCols = 512;
constexpr int kTSCol = 0;                   // S^T buffers: 2 x 32 columns
constexpr int kTOCol = 64;                  // O^T buffers: 2 x 32 columns
constexpr int kTVCol = 128;                 // V^T buffers: 2 x 64 columns (128 tokens, two bf16 per column)
constexpr int kTOLoCol = 256;               // O^T of the P residuals: 2 x 32 columns
constexpr int kTPHalf = 128 * kTN * 2;      // P^T high part (then the residual): [128 tokens][32 queries] bf16

template <int D>
__host__ __device__ constexpr int t_karea() { return kTPages * kPage * D * 2; }  // a group's K, then its P^T
template <int D>
__host__ __device__ constexpr int t_slot() { return 2 * t_karea<D>(); }          // K area, then V area
template <int D>
__host__ __device__ constexpr int t_qbuf() { return D / 64 * kTN * 128; }        // Q: [D/64 halves][32 rows][128 B]

struct TLayout {
  int ring, q, flags, wmax, lw, mfin, mref, gpre, plen, desc, rowbits, slen, total;
};

// Shared-memory carve-up (identical on host and device); the ring and the Q
// buffers are 1024-byte aligned (128-byte swizzle atoms).
template <int D>
__host__ __device__ inline TLayout t_layout(int nslots, int G, int R) {
  TLayout L;
  L.ring = 0;
  L.q = nslots * t_slot<D>();
  L.flags = L.q + 2 * t_qbuf<D>();      // [4 sets][2][4] int: a softmax warp needs the maxima moved
  L.wmax = L.flags + 32 * 4;            // [4][32] per-quarter query maxima of a group
  L.lw = L.wmax + 4 * kTN * 4;          // [2 pieces][4][32] per-warp query sums
  L.mfin = L.lw + 2 * 4 * kTN * 4;      // [2 pieces][32] query reference maxima at the piece end
  L.mref = L.mfin + 2 * kTN * 4;        // [2 versions][32] current query reference maxima
  L.gpre = L.mref + 2 * kTN * 4;
  L.plen = align_up(L.gpre + (G + 1) * 4, 16);
  L.desc = align_up(L.plen + G * 4, 16);
  L.rowbits = align_up(L.desc + nslots * kTPages * 4, 16);
  L.slen = align_up(L.rowbits + (R + 31) / 32 * 4, 16);
  L.total = align_up(L.slen + R * 4, 16) + 1024;  // + slack for the 1024-byte aligned base
  return L;
}

// 64-byte swizzle of a [rows][64 B] tile (16-byte chunk index XOR bits 1-2 of the row).
__device__ __forceinline__ uint32_t sw64_off(int row, int chunk) {
  return (uint32_t)(row * 64 + (((chunk ^ (row >> 1)) & 3) << 4));
}
// 128-byte swizzle of a [rows][128 B] tile (16-byte chunk index XOR the row mod 8).
__device__ __forceinline__ uint32_t sw128_off(int row, int chunk) {
  return (uint32_t)(row * 128 + (((chunk ^ row) & 7) << 4));
}

// Warp reduction of 32 values per lane over the lanes, ending with lane L
// holding the result for index L: at each step a lane keeps the half of its
// values on its side of the partner bit and receives the partner's copies of
// that half (31 shuffles instead of 32 x 5).
template <typename Op>
__device__ __forceinline__ float transpose_reduce32(float (&v)[32], int lane, Op op) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float send = up ? v[i] : v[i + o];
      const float keep = up ? v[i + o] : v[i];
      v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, o));
    }
  }
  return v[0];
}

// The same for 16 values per lane: one butterfly step over the lane halves,
// then halving over 16 lanes; lane L ends with the result for index L & 15.
template <typename Op>
__device__ __forceinline__ float transpose_reduce16(float (&v)[16], int lane, Op op) {
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = op(v[i], __shfl_xor_sync(0xffffffffu, v[i], 16));
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float send = up ? v[i] : v[i + o];
      const float keep = up ? v[i + o] : v[i];
      v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, o));
    }
  }
  return v[0];
}

// The same for 8 values per lane: two butterfly steps over the lane quarters,
// then halving over 8 lanes; lane L ends with the result for index L & 7.
template <typename Op>
__device__ __forceinline__ float transpose_reduce8(float (&v)[8], int lane, Op op) {
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = op(v[i], __shfl_xor_sync(0xffffffffu, v[i], 16));
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = op(v[i], __shfl_xor_sync(0xffffffffu, v[i], 8));
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    const bool up = (lane & o) != 0;
#pragma unroll
    for (int i = 0; i < o; ++i) {
      const float send = up ? v[i] : v[i + o];
      const float keep = up ? v[i + o] : v[i];
      v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, o));
    }
  }
  return v[0];
}

// P = hi + lo with hi = p truncated to bf16 and lo = (p - hi) truncated to bf16
// (|p - hi - lo| <= 2^-16 |p|), two values per 32-bit word, the first in the
// low half.
__device__ __forceinline__ void split_bf16x2(float p0, float p1, uint32_t& hi, uint32_t& lo) {
  const uint32_t h0 = __float_as_uint(p0) & 0xffff0000u, h1 = __float_as_uint(p1) & 0xffff0000u;
  const uint32_t l0 = __float_as_uint(p0 - __uint_as_float(h0)), l1 = __float_as_uint(p1 - __uint_as_float(h1));
  hi = (h0 >> 16) | h1;
  lo = (l0 >> 16) | (l1 & 0xffff0000u);
}

template <int D, int NS>
__global__ void __launch_bounds__(t_threads<NS>(), 1)
    attn_t_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const AttnParams p) {
  constexpr int kTile = kPage * D * 2;  // one K or V page-head tile
  constexpr int kStage = 2 * kTile;     // bytes one page brings in
  constexpr int kHalves = D / 64;
  constexpr int kKArea = t_karea<D>();
  constexpr int kSlot = t_slot<D>();
  constexpr int kQBuf = t_qbuf<D>();
  constexpr int kThr = t_threads<NS>();
  constexpr uint32_t kIdQK = idesc_bf16_f32(128, kTN, 0, 0);  // A = K, B = Q: both K-major
  constexpr uint32_t kIdPV = idesc_bf16_f32(128, kTN, 0, 1);  // A = V^T from TMEM, B = P^T MN-major
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const TLayout L = t_layout<D>(p.nslots, p.G, p.G * p.rpg);
  uint32_t* rowbits = reinterpret_cast<uint32_t*>(smem + L.rowbits);
  int32_t* gpre = reinterpret_cast<int32_t*>(smem + L.gpre);
  int32_t* plen_s = reinterpret_cast<int32_t*>(smem + L.plen);
  int32_t* slen_s = reinterpret_cast<int32_t*>(smem + L.slen);
  uint32_t* descs = reinterpret_cast<uint32_t*>(smem + L.desc);
  __shared__ uint64_t full_bar[kTMaxSlots], empty_bar[kTMaxSlots];
  __shared__ uint64_t s_full[2], s_empty[2], p_full[2], p_empty[2], q_full[2], q_empty[2];
  __shared__ uint64_t o_full[2], o_free[2], ml_full[2], ml_empty[2], mma_done[3];
  __shared__ int32_t s_abort, s_issued, s_tick, s_wsum[kThr / 32];
  __shared__ uint32_t s_tmem;
  __shared__ PieceIter s_it;
  volatile int32_t* abort_flag = &s_abort;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int c = blockIdx.x;
  const int ns = p.nslots;
  const uint32_t sbase = smem_u32(smem);
  const int nrows = p.G * p.rpg;

  if (tid == 0) {
    for (int i = 0; i < ns; ++i) {
      mbar_init(&full_bar[i], kTPages);  // one arrival per page position (absent pages of a short group too)
      mbar_init(&empty_bar[i], 2);       // the group's two PV commits
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], 4 * NS);
      mbar_init(&p_full[i], 4 * NS);
      mbar_init(&p_empty[i], 2);
      mbar_init(&q_full[i], 4);
      mbar_init(&q_empty[i], 1);
      mbar_init(&o_full[i], 2);
      mbar_init(&o_free[i], 4);
      mbar_init(&ml_full[i], 4 * NS);
      mbar_init(&ml_empty[i], 4);
      mbar_init(&mma_done[i], 1);
    }
    mbar_init(&mma_done[2], 1);
    s_abort = 0;
    s_issued = 0;
    fence_mbar_init();
  }
  if (warp == kTQk) {
    tmem_alloc(&s_tmem, kTTmemCols);
    tmem_relinquish();
  }
  if (warp == kTProd && lane == 0) {  // the copies' descriptors, fetched while the set-up runs
    prefetch_tensormap(&tmK);
    prefetch_tensormap(&tmV);
  }
  // This block's share of the block tables and queries is asked of L2 while the
  // lengths load (each line once over the grid), so that the first block-table
  // and query loads of every block find them there.
  {
    const int64_t nb_p = (int64_t)p.G * p.max_pp * 4, nb_s = (int64_t)nrows * p.max_sp * 4;
    const int64_t nb_q = (int64_t)nrows * p.Hq * D * 2;
    const int64_t lp = (nb_p + 127) / 128, ls = (nb_s + 127) / 128, lq = (nb_q + 127) / 128;
    const int64_t step = (int64_t)p.C * kThr;
    for (int64_t l = (int64_t)tid * p.C + c; l < lp + ls + lq; l += step) {
      if (l < lp) prefetch_l2(reinterpret_cast<const uint8_t*>(p.prompt_bt) + l * 128);
      else if (l < lp + ls) prefetch_l2(reinterpret_cast<const uint8_t*>(p.suffix_bt) + (l - lp) * 128);
      else prefetch_l2(reinterpret_cast<const uint8_t*>(p.q) + (l - lp - ls) * 128);
    }
  }
  // ---- lengths and activity flags, all loads issued together, kept in shared memory ----
  for (int r0 = warp * 32; r0 < max(nrows, p.G); r0 += kThr) {  // (whole warps: the ballot below)
    const int r = r0 + lane;
    int act = 0, sl = 0, pl = 0;
    if (r < nrows) {
      act = p.row_active == nullptr ? 1 : p.row_active[r];
      sl = p.suffix_len[r];
    }
    if (r < p.G) pl = p.prompt_len[r];
    if (r < nrows) {
      if (c == 0 && (sl < 0 || sl > p.max_sp * kPage)) flag(p.dev_status, RGD_DEV_BAD_PAGE);
      slen_s[r] = act ? clamp_len(sl, p.max_sp) : 0;
    }
    if (r < p.G) {
      if (c == 0 && (pl < 0 || pl > p.max_pp * kPage)) flag(p.dev_status, RGD_DEV_BAD_PAGE);
      plen_s[r] = clamp_len(pl, p.max_pp);
    }
    const uint32_t bits = __ballot_sync(0xffffffffu, r < nrows && act != 0);
    if (lane == 0 && r0 < nrows) rowbits[r0 >> 5] = bits;
  }
  if (tid == 0) gpre[0] = 0;
  __syncthreads();
  // a group's pages: its prompt pages if any row of it is active, plus its
  // active rows' suffix pages
  for (int g = tid; g < p.G; g += kThr) {
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
  if (p.G <= 32) {  // inclusive prefix sum of gpre[1..G]: one warp (uniform branch)
    if (warp == 0) {
      int incl = lane < p.G ? gpre[lane + 1] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      if (lane < p.G) gpre[lane + 1] = incl;
    }
  } else {  // the same over every thread
    const int E = (p.G + kThr - 1) / kThr;
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
      for (int w = 0; w < kThr / 32; ++w) {
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
  const int Ceff = (int)min((int64_t)p.C, T);
  const int64_t b = c < Ceff ? div_nn((int64_t)c * T, Ceff) : T;
  const int64_t e = c < Ceff ? div_nn((int64_t)(c + 1) * T, Ceff) : T;
  if (tid == 0 && b < e) s_it = piece_iter(p, gpre, b, e);
  __syncthreads();

  if (warp == kTProd) {
    // ============================ producers ===========================
    // One warp, 32 pages (one per lane) a round, groups of 8 pages: K halves
    // land half-major ([D/64][8 pages][16 rows][128 B], so that a group's K is
    // one 128-row A operand per half), V tiles page-major after them.  A round's
    // pages are resolved (job by binary search, then the block-table entry)
    // before the previous round's copies wait for their slots, so the
    // block-table loads are in flight while the warp waits.
    if (b < e) {
      const uint64_t pol = policy_evict_first();
      const PieceIter& it = s_it;
      struct Pg {
        int32_t page, tok, rowsel, hh, jpos, ng;
        bool valid;
      };
      auto resolve = [&](int64_t ib) {
        Pg r{-1, 0, -1, 0, 0, 0, ib + lane < e - b};
        if (r.valid) {
          const int64_t x = seq_page(it, b, ib + lane);
          const Job jb = job_at(p, gpre, x);
          // this block's piece of the job starts at max(b, job start); groups restart there
          const int64_t pstart = max(b, jb.start);
          const int kin = (int)(x - pstart);
          const int npiece = (int)(min(e, jb.start + jb.n) - pstart);
          r.jpos = kin % kTPages;
          r.ng = min(kTPages, npiece - (kin - r.jpos));
          const int k = (int)(x - jb.start);
          const int plen = plen_s[jb.g];
          const int ppg = (plen + kPage - 1) / kPage;
          r.hh = jb.h;
          if (k < ppg) {
            r.page = __ldg(p.prompt_bt + (int64_t)jb.g * p.max_pp + k);
            r.tok = min(kPage, plen - k * kPage);
          } else {
            int ks = k - ppg;
            for (int rr = 0; rr < p.rpg; ++rr) {  // the active row holding suffix page ks
              const int r2 = jb.g * p.rpg + rr;
              const int slen = slen_s[r2];
              const int np = (slen + kPage - 1) / kPage;
              if (ks < np) {
                r.page = __ldg(p.suffix_bt + (int64_t)r2 * p.max_sp + ks);
                r.tok = min(kPage, slen - ks * kPage);
                r.rowsel = rr;
                break;
              }
              ks -= np;
            }
          }
        }
        return r;
      };
      int gbase = 0;  // groups started before sequence position ib
      Pg cur = resolve(0);
      for (int64_t ib = 0; ib < e - b; ib += 32) {
        const Pg nxt = resolve(ib + 32);  // (loads in flight during this round's waits)
        const bool start = cur.valid && cur.jpos == 0;
        const uint32_t starts = __ballot_sync(0xffffffffu, start);
        const uint32_t le = 0xffffffffu >> (31 - lane);
        const int gidx = gbase + __popc(starts & le) - 1;  // lane 0 may continue the last round's group
        const int g0 = __shfl_sync(0xffffffffu, gidx, 0);
        const int g1 = __shfl_sync(0xffffffffu, gidx, 31 - __clz(__ballot_sync(0xffffffffu, cur.valid)));
        const int gs = gidx % ns;
        bool aborted = false;
        for (int gq = g0; gq <= g1; ++gq) {
          const bool in = cur.valid && gidx == gq;
          const bool lead = in && (start || lane == 0);
          int stop = 0;
          if (lead && gq >= ns &&
              !wait_or_abort(&empty_bar[gs], (uint32_t)((gq / ns) - 1) & 1u, abort_flag, p.wait_ns))
            stop = 1;
          if (__any_sync(0xffffffffu, stop != 0)) {
            aborted = true;
            break;
          }
          if (in) {
            int32_t y = -2 * kPage;  // fully out of bounds: the TMA fills zeros
            if (cur.page >= 0 && cur.page < p.num_pages) y = (cur.page * p.Hkv + cur.hh) * kPage;
            else flag(p.dev_status, RGD_DEV_BAD_PAGE);
            descs[gs * kTPages + cur.jpos] = (uint32_t)cur.tok | ((uint32_t)(cur.rowsel & 0xffff) << 16);
            uint8_t* sl = smem + gs * kSlot;
            mbar_arrive_expect_tx(&full_bar[gs], kStage);
            if (cur.jpos == cur.ng - 1 && cur.ng < kTPages) mbar_arrive_cnt(&full_bar[gs], kTPages - cur.ng);
#pragma unroll
            for (int hf = 0; hf < kHalves; ++hf)
              tma_load_3d_hint(sl + hf * (kTPages * 2048) + cur.jpos * 2048, &tmK, &full_bar[gs], 0, y, hf, pol);
            tma_load_3d_hint(sl + kKArea + cur.jpos * kTile, &tmV, &full_bar[gs], 0, y, 0, pol);
            if (start) atomicMax(&s_issued, gq + 1);
          }
        }
        if (aborted) break;
        gbase += __popc(starts);
        cur = nxt;
      }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  } else if (warp == kTQk) {
    // ============================ QK issue ============================
    if (lane == 0 && b < e) {
      const uint64_t kdesc = smem_desc(sbase, 16, 1024, 2);
      const uint64_t qdesc = smem_desc(sbase + L.q, 16, 1024, 2);
      int gi = 0, pc = 0;
      bool ok = true;
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      for (bool more = true; ok && more; more = next_piece(p, gpre, it, pc, cur, n_in)) {
        const int qb = pc & 1;
        if (!wait_or_abort(&q_full[qb], (uint32_t)(pc >> 1) & 1u, abort_flag, p.wait_ns)) break;
        for (int k0 = 0; k0 < n_in; k0 += kTPages) {
          const int sb = gi & 1, gs = gi % ns;
          if (!wait_or_abort(&full_bar[gs], (uint32_t)(gi / ns) & 1u, abort_flag, p.wait_ns) ||
              (gi >= 2 && !wait_or_abort(&s_empty[sb], (uint32_t)((gi >> 1) - 1) & 1u, abort_flag, p.wait_ns))) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t a = kdesc + (uint64_t)((gs * kSlot + (kk >> 2) * (kTPages * 2048) + (kk & 3) * 32) >> 4);
            const uint64_t bq = qdesc + (uint64_t)((qb * kQBuf + (kk >> 2) * (kTN * 128) + (kk & 3) * 32) >> 4);
            umma_bf16(tmem + kTSCol + sb * kTN, a, bq, kIdQK, kk > 0 ? 1u : 0u);
          }
          umma_commit(&s_full[sb]);
          if (k0 + kTPages >= n_in) umma_commit(&q_empty[qb]);  // Q's buffer may take the piece after next
          ++gi;
        }
        ++pc;
      }
    }
  } else if (warp == kTPv || warp == kTPvLo) {
    // ============================ PV issue ============================
    // warp kTPv: the P high parts into O^T; warp kTPvLo: the residuals into
    // the second O^T (both read V^T and their P^T part of the group)
    const bool lo = warp == kTPvLo;
    if (lane == 0 && b < e) {
      const uint64_t pdesc = smem_desc(sbase, 8192, 512, 4);  // P^T: MN-major, 64-byte swizzle
      int gi = 0, pc = 0;
      bool ok = true;
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      for (bool more = true; ok && more; more = next_piece(p, gpre, it, pc, cur, n_in)) {
        const uint32_t od = tmem + (lo ? kTOLoCol : kTOCol) + (pc & 1) * kTN;
        for (int k0 = 0; k0 < n_in; k0 += kTPages) {
          const int ng = min(kTPages, n_in - k0);
          const int pb = gi & 1, gs = gi % ns;
          if (!wait_or_abort(&p_full[pb], (uint32_t)(gi >> 1) & 1u, abort_flag, p.wait_ns) ||
              (k0 == 0 && pc >= 2 &&
               !wait_or_abort(&o_free[pc & 1], (uint32_t)((pc >> 1) - 1) & 1u, abort_flag, p.wait_ns))) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int j = 0; j < kTPages; ++j) {
            if (j < ng) {
              const uint32_t a = tmem + kTVCol + pb * 64 + j * 8;  // page j's 16 tokens of V^T
              const uint64_t pd = pdesc + (uint64_t)((gs * kSlot + (lo ? kTPHalf : 0) + j * 1024) >> 4);
              umma_bf16_tmem_a(od, a, pd, kIdPV, (k0 == 0 && j == 0) ? 0u : 1u);
            }
          }
          umma_commit(&p_empty[pb]);
          umma_commit(&empty_bar[gs]);  // the slot's V and P^T are no longer read
          if (k0 + kTPages >= n_in) umma_commit(&o_full[pc & 1]);
          ++gi;
        }
        ++pc;
      }
    }
  } else if (warp < kTEpi || warp >= kTSoftB) {
    // ============================ softmax ============================
    // Thread = token t of the group (lane quarter qd); set hs takes queries
    // 8hs..8hs+7.  The reference maxima of the queries (log2 units) live in
    // shared memory, two versions: a group that moves a set's maxima writes the
    // other version and the set's threads switch after a barrier, so all use
    // the same reference for a group.  lacc[i] is this thread's running sum of
    // query 8hs + i.  Before its scores, each thread copies V^T for head
    // dimension 32qd + lane and the set's pages of the group into TMEM.
    const int qd = warp & 3, hs = warp < 4 ? 0 : 1 + (warp - kTSoftB) / 4;
    const int t = qd * 32 + lane, jp = t >> 4, tip = t & 15;
    const int q0 = hs * kTQS;
    const uint32_t tl = tmem + ((uint32_t)(qd * 32) << 16);
    int32_t* flags = reinterpret_cast<int32_t*>(smem + L.flags) + hs * 8;
    float* wmax = reinterpret_cast<float*>(smem + L.wmax);
    float* lw = reinterpret_cast<float*>(smem + L.lw);
    float* mfin = reinterpret_cast<float*>(smem + L.mfin);
    float* mref_s = reinterpret_cast<float*>(smem + L.mref);  // [2 versions][32]
    // named barrier of the set's 128 threads (0 is __syncthreads, 2 the piece ends')
    auto set_sync = [&]() { asm volatile("bar.sync %0, 128;" ::"r"(hs == 0 ? 1 : hs + 2) : "memory"); };
    auto wwait = [&](uint64_t* bar, uint32_t parity) {
      return __all_sync(0xffffffffu, wait_or_abort(bar, parity, abort_flag, p.wait_ns));
    };
    const uint32_t qall = p.nq >= 32 ? 0xffffffffu : ((1u << p.nq) - 1u);
    const uint32_t growmask = p.gq >= 32 ? 0xffffffffu : ((1u << p.gq) - 1u);
    // V^T copy: this thread's head dimension and its byte within the swizzled V rows
    const int dv = qd * 32 + lane;
    const int vchunk = ((dv & 63) * 2) >> 4;
    const uint32_t voff = (uint32_t)((dv >> 6) * 2048 + (((dv & 63) * 2) & 15));
    float lacc[kTQS];
#pragma unroll
    for (int i = 0; i < kTQS; ++i) lacc[i] = 0.f;
    int mv = 0;          // current version of the reference maxima
    bool fresh = true;   // piece start: every reference is -inf (not read from shared memory)
    int gi = 0;
    bool ok = true;
    if (b < e) {
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      int pc = 0;
      for (bool more = true; more; more = next_piece(p, gpre, it, pc, cur, n_in)) {
        const int ob = pc & 1;
        for (int k0 = 0; k0 < n_in; k0 += kTPages) {
          const int ng = min(kTPages, n_in - k0);
          const int sb = gi & 1, gs = gi % ns;
          const bool has = jp < ng;
          if (ok && !wwait(&full_bar[gs], (uint32_t)(gi / ns) & 1u)) ok = false;
          // the PV two groups back has read this group's V^T buffer (and taken its P barrier phase)
          if (gi >= 2 && ok && !wwait(&p_empty[sb], (uint32_t)((gi >> 1) - 1) & 1u)) ok = false;
          if (ok && dv < D) {
            const uint32_t vb = sbase + gs * kSlot + kKArea + voff;
            tc_fence_after();
#pragma unroll
            for (int k = 0; k < (kTPages + NS - 1) / NS; ++k) {
              const int jj = hs + k * NS;  // a page of the group: tokens 16jj..16jj+15
              if (jj < kTPages) {
                uint32_t vt[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                  const int r = 2 * i;
                  const uint32_t a0 = vb + jj * kTile + r * 128 + (((vchunk ^ r) & 7) << 4);
                  const uint32_t a1 = vb + jj * kTile + (r + 1) * 128 + (((vchunk ^ (r + 1)) & 7) << 4);
                  uint16_t x0, x1;
                  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(x0) : "r"(a0));
                  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(x1) : "r"(a1));
                  vt[i] = (uint32_t)x0 | ((uint32_t)x1 << 16);
                }
                tmem_st8(tl + kTVCol + sb * 64 + jj * 8, vt);
              }
            }
          }
          int tok = 0, sel = -1;
          if (ok && has) {
            const uint32_t dsc = descs[gs * kTPages + jp];
            tok = (int)(dsc & 0xffffu);
            sel = (int)(int16_t)(dsc >> 16);
          }
          if (ok && !wwait(&s_full[sb], (uint32_t)(gi >> 1) & 1u)) ok = false;
          tc_fence_after();
          float sc[kTQS];
          if (ok) {
            tmem_ld8(tl + kTSCol + sb * kTN + q0, reinterpret_cast<uint32_t(&)[kTQS]>(sc));
            tmem_ld_wait();
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&s_empty[sb]);  // S^T is in registers
          // visible queries of this token: the job's nq, and for a suffix page
          // only the queries of the row that owns it
          uint32_t vis = 0;
          if (ok && has && tip < tok) vis = sel < 0 ? qall : (qall & (growmask << (sel * p.gq)));
          vis >>= q0;
          const float* mr = mref_s + mv * kTN + q0;
          bool ex = false;
#pragma unroll
          for (int q = 0; q < kTQS; q += 4) {
            const float4 m4 = fresh ? make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY)
                                    : *reinterpret_cast<const float4*>(mr + q);
            const float mm[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              sc[q + u] = ((vis >> (q + u)) & 1u) ? sc[q + u] * p.scale_log2 : -INFINITY;
              ex = ex || (sc[q + u] > mm[u] + kRescaleLog2);
            }
          }
          // do the set's reference maxima move for this group? (its four warps agree)
          int32_t* fl = flags + (gi & 1) * 4;
          const bool wany = __any_sync(0xffffffffu, ex);
          if (lane == 0) fl[qd] = wany ? 1 : 0;
          set_sync();
          if ((fl[0] | fl[1] | fl[2] | fl[3]) != 0) {
            // this warp's query maxima (lane i: query q0 + i), then the new
            // reference of each query from the four warps and its factor f
            float v[kTQS];
#pragma unroll
            for (int q = 0; q < kTQS; ++q) v[q] = sc[q];
            const float wm = transpose_reduce8(v, lane, [](float x, float y) { return fmaxf(x, y); });
            if (lane < kTQS) wmax[qd * kTN + q0 + lane] = wm;
            set_sync();
            const int qi = q0 + (lane & (kTQS - 1));
            const float mo = fresh ? -INFINITY : mr[lane & (kTQS - 1)];
            const float mn = fmaxf(fmaxf(mo, wmax[qi]), fmaxf(fmaxf(wmax[kTN + qi], wmax[2 * kTN + qi]),
                                                             wmax[3 * kTN + qi]));
            const float fq = mo == -INFINITY ? 0.f : exp2f(mo - mn);
            if (qd == 0 && lane < kTQS) mref_s[(mv ^ 1) * kTN + qi] = mn;
#pragma unroll
            for (int q = 0; q < kTQS; ++q) lacc[q] *= __shfl_sync(0xffffffffu, fq, q);
            // O^T already holds this piece's earlier groups: once their PV is
            // done, the set's query columns (this warp's 32 head dimensions) are scaled
            if (k0 > 0) {
              const int pg = gi - 1;
              if (ok && !wwait(&p_empty[pg & 1], (uint32_t)(pg >> 1) & 1u)) ok = false;
              if (ok) {
                tc_fence_after();
#pragma unroll
                for (int part = 0; part < 2; ++part) {
                  const uint32_t oc = tl + (part ? kTOLoCol : kTOCol) + ob * kTN + q0;
                  uint32_t o8[kTQS];
                  tmem_ld8(oc, o8);
                  tmem_ld_wait();
#pragma unroll
                  for (int u = 0; u < kTQS; ++u)
                    o8[u] = __float_as_uint(__uint_as_float(o8[u]) * __shfl_sync(0xffffffffu, fq, u));
                  tmem_st8(oc, o8);
                }
              }
            }
            set_sync();  // the new version is written, wmax and the old version are read
            mv ^= 1;
            fresh = false;
          }
          // P = 2^(s - m) in bf16 high part + residual (ex2 of -inf is +0)
          uint32_t ph[kTQS / 2], plo[kTQS / 2];
          const float* mc = mref_s + mv * kTN + q0;
#pragma unroll
          for (int q = 0; q < kTQS; q += 4) {
            const float4 m4 = fresh ? make_float4(0.f, 0.f, 0.f, 0.f) : *reinterpret_cast<const float4*>(mc + q);
            const float mm[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll
            for (int u = 0; u < 4; u += 2) {
              const float r0 = mm[u] == -INFINITY ? 0.f : mm[u];
              const float r1 = mm[u + 1] == -INFINITY ? 0.f : mm[u + 1];
              const float p0 = ex2_approx(sc[q + u] - r0), p1 = ex2_approx(sc[q + u + 1] - r1);
              lacc[q + u] += p0;
              lacc[q + u + 1] += p1;
              split_bf16x2(p0, p1, ph[(q + u) / 2], plo[(q + u) / 2]);
            }
          }
          // the group's slot is the P^T area once its QK is done (this set's 16 bytes of each row)
          if (ok) {
            const uint32_t pbase = sbase + gs * kSlot;
            st_shared_v4(pbase + sw64_off(t, hs), ph[0], ph[1], ph[2], ph[3]);
            st_shared_v4(pbase + kTPHalf + sw64_off(t, hs), plo[0], plo[1], plo[2], plo[3]);
          }
          tmem_st_wait();            // V^T (and any O rescale) are in TMEM
          fence_proxy_async_smem();  // the MMAs read P^T through the async proxy
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&p_full[sb]);
          ++gi;
        }
        // piece end: per-warp query sums and the reference maxima to the epilogue warps
        if (pc >= 2 && ok && !wwait(&ml_empty[ob], (uint32_t)((pc >> 1) - 1) & 1u)) ok = false;
        const float ls = transpose_reduce8(lacc, lane, [](float x, float y) { return x + y; });
        if (lane < kTQS) {
          lw[(ob * 4 + qd) * kTN + q0 + lane] = ls;
          if (qd == 0) mfin[ob * kTN + q0 + lane] = fresh ? -INFINITY : mref_s[mv * kTN + q0 + lane];
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&ml_full[ob]);
#pragma unroll
        for (int q = 0; q < kTQS; ++q) lacc[q] = 0.f;
        fresh = true;
        ++pc;
      }
    }
  } else {
    // ============================ piece ends ==========================
    // Thread = head dimension d of O^T (lane quarter w).  Writes Q of the
    // pieces two ahead, reads a finished piece's O^T, and writes the output,
    // the partial of a split job, or -- in a merger -- the merged output.
    const int w = warp - kTEpi;
    const int d = w * 32 + lane;
    const int et = w * 32 + lane;  // index among the 128 epilogue threads
    const uint32_t tl = tmem + ((uint32_t)(w * 32) << 16);
    const float* lw = reinterpret_cast<const float*>(smem + L.lw);
    const float* mfin = reinterpret_cast<const float*>(smem + L.mfin);
    auto epi_sync = [&]() { asm volatile("bar.sync 2, 128;" ::: "memory"); };
    auto wwait = [&](uint64_t* bar, uint32_t parity) {
      return __all_sync(0xffffffffu, wait_or_abort(bar, parity, abort_flag, p.wait_ns));
    };
    const int nq = p.nq, gq = p.gq;
    bool ok = true;
    // Q of job jb into Q buffer qb: [D/64 halves][32 rows][128 B], 128-byte swizzle; rows >= nq are zero
    auto write_q = [&](const Job& jb, int qb) {
      constexpr int kCh = D / 8;  // 16-byte chunks per query row
      const uint32_t qbase = sbase + L.q + qb * kQBuf;
#pragma unroll 1
      for (int idx = et; idx < kTN * kCh; idx += 128) {
        const int q = idx / kCh, cc = idx % kCh;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (q < nq) {
          const int rr = jb.g * p.rpg + q / gq, hq = jb.h * gq + q % gq;
          v = __ldg(reinterpret_cast<const uint4*>(p.q + ((int64_t)rr * p.Hq + hq) * D) + cc);
        }
        st_shared_v4(qbase + (cc >> 3) * (kTN * 128) + sw128_off(q, cc & 7), v.x, v.y, v.z, v.w);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&q_full[qb]);
    };
    // jobs with no pages at all (empty prompt and suffixes, some row active)
    for (int j = c; j < p.G * p.Hkv; j += p.C) {
      const int g = j / p.Hkv, h = j % p.Hkv;
      if (gpre[g + 1] != gpre[g]) continue;
      for (int idx = et; idx < nq * D; idx += 128) {
        const int i = idx / D, dd = idx % D;
        const int rr = g * p.rpg + i / gq, hq = h * gq + i % gq;
        if (!row_on(p, rr)) continue;
        p.out[((int64_t)rr * p.Hq + hq) * D + dd] = __float2bfloat16(0.f);
        if (dd == 0 && p.lse) p.lse[(int64_t)rr * p.Hq + hq] = -INFINITY;
      }
    }
    if (b < e) {
      const PieceIter& it = s_it;
      Job cur = it.j0;
      int n_in = it.n0;
      // Q of the first two pieces
      Job nx1 = cur, nx2 = cur;
      int n1 = n_in, n2 = n_in;
      bool has1 = next_piece(p, gpre, it, 1, nx1, n1);
      write_q(cur, 0);
      if (has1) write_q(nx1, 1);
      nx2 = nx1;
      n2 = n1;
      bool has2 = has1 && next_piece(p, gpre, it, 2, nx2, n2);
      for (int pc = 0;; ++pc) {
        const int ob = pc & 1;
        const int j = cur.g * p.Hkv + cur.h;
        const int first = cta_of(cur.start, T, Ceff), last = cta_of(cur.start + cur.n - 1, T, Ceff);
        const bool split = first != last;
        const int nparts = last - first;
        const bool merger = split && c == first;
        // ---- this piece's O^T row (head dim d), and per lane q the maxima,
        // sum and output row of query q ----
        if (ok && !wwait(&o_full[ob], (uint32_t)(pc >> 1) & 1u)) ok = false;
        if (ok && !wwait(&ml_full[ob], (uint32_t)(pc >> 1) & 1u)) ok = false;
        tc_fence_after();
        uint32_t ov[kTN];
        if (ok) {
          uint32_t ol[kTN];
          tmem_ld32(tl + kTOCol + ob * kTN, ov);
          tmem_ld32(tl + kTOLoCol + ob * kTN, ol);
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < kTN; ++q) ov[q] = __float_as_uint(__uint_as_float(ov[q]) + __uint_as_float(ol[q]));
        }
        float Ml = -INFINITY, Ll = 0.f;
        int orow = -1;  // rr * Hq + hq of query `lane` if its row is active
        if (lane < nq) {
          Ml = mfin[ob * kTN + lane];
          Ll = (lw[(ob * 4) * kTN + lane] + lw[(ob * 4 + 1) * kTN + lane]) +
               (lw[(ob * 4 + 2) * kTN + lane] + lw[(ob * 4 + 3) * kTN + lane]);
          const int rr = cur.g * p.rpg + lane / gq, hq = cur.h * gq + lane % gq;
          if ((rowbits[rr >> 5] >> (rr & 31)) & 1u) orow = rr * p.Hq + hq;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&o_free[ob]);
          mbar_arrive(&ml_empty[ob]);
        }
        const bool out_ok = __all_sync(0xffffffffu, ok && !*abort_flag);
        const int64_t s_idx = (int64_t)c + j;
        const int mls = ml_stride(nq);
        if (split && !merger) {
          // this piece's partial (unnormalised O and (M, L) per query), then its count
          if (out_ok && d < D) {
#pragma unroll
            for (int q = 0; q < kTN; ++q)
              if (q < nq) p.slot_o[(s_idx * nq + q) * D + d] = __uint_as_float(ov[q]);
          }
          if (out_ok && w == 0 && lane < nq) p.slot_ml[s_idx * mls + lane] = make_float2(Ml, Ll);
          __threadfence();
          epi_sync();
          if (et == 0) atomicAdd(p.ticket + j, out_ok && !*abort_flag ? 1 : 0x10001);
        } else {
          bool good = out_ok;
          if (merger) {
            // wait for the job's other pieces (each the first piece of its block,
            // never behind a wait on this one), then fold their partials in
            if (et == 0) {
              const uint64_t t0 = globaltimer_ns();
              int tk = 0;
              for (;;) {
                tk = ld_acquire_gpu(p.ticket + j);
                if ((tk & 0xffff) == nparts) break;
                if (*abort_flag || globaltimer_ns() - t0 > p.wait_ns) {
                  *abort_flag = 1;
                  tk = -1;
                  break;
                }
                __nanosleep(128);
              }
              s_tick = tk;
            }
            epi_sync();
            good = good && s_tick > 0 && (s_tick >> 16) == 0;
            if (good) {
              __threadfence();
              if (!(Ll > 0.f)) Ml = -INFINITY;  // (a piece that saw none of the query's tokens)
#pragma unroll 1
              for (int k = 0; k < nparts; ++k) {
                const int64_t sl = (int64_t)(first + k + 1) + j;
                const float2 mlk = lane < nq ? p.slot_ml[sl * mls + lane] : make_float2(-INFINITY, 0.f);
                float po[kTN];
#pragma unroll
                for (int q = 0; q < kTN; ++q) po[q] = (q < nq && d < D) ? p.slot_o[(sl * nq + q) * D + d] : 0.f;
                // lane q: the weights of query q's running result and of this partial
                float fa = 1.f, fb = 0.f;
                if (mlk.y > 0.f) {
                  const float mn = fmaxf(Ml, mlk.x);
                  fa = Ml == -INFINITY ? 0.f : exp2f(Ml - mn);
                  fb = exp2f(mlk.x - mn);
                  Ll = Ll * fa + mlk.y * fb;
                  Ml = mn;
                }
#pragma unroll
                for (int q = 0; q < kTN; ++q)
                  ov[q] = __float_as_uint(__uint_as_float(ov[q]) * __shfl_sync(0xffffffffu, fa, q) +
                                          po[q] * __shfl_sync(0xffffffffu, fb, q));
              }
            }
          }
          if (good) {
            const float inv = Ll > 0.f ? 1.f / Ll : 0.f;
#pragma unroll
            for (int q = 0; q < kTN; ++q) {
              const float iv = __shfl_sync(0xffffffffu, inv, q);
              const int orq = __shfl_sync(0xffffffffu, orow, q);
              if (q < nq && orq >= 0 && d < D)
                p.out[(int64_t)orq * D + d] = __float2bfloat16(__uint_as_float(ov[q]) * iv);
            }
            if (p.lse && w == 0 && orow >= 0) p.lse[orow] = Ll > 0.f ? (Ml + log2f(Ll)) * kLn2 : -INFINITY;
          }
          if (merger) {
            epi_sync();
            if (et == 0) p.ticket[j] = 0;  // every other piece has counted itself
          }
        }
        // ---- Q of the piece two ahead, into this piece's Q buffer ----
        if (has2) {
          if (ok && !wwait(&q_empty[ob], (uint32_t)(pc >> 1) & 1u)) ok = false;
          if (ok) write_q(nx2, ob);
          else if (lane == 0) mbar_arrive(&q_full[ob]);  // (keeps the QK warp's waits bounded by the abort)
        }
        if (!has1) break;
        cur = nx1;
        n_in = n1;
        nx1 = nx2;
        n1 = n2;
        has1 = has2;
        if (has2) has2 = next_piece(p, gpre, it, pc + 3, nx2, n2);
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
    }
    if ((warp == kTQk || warp == kTPv || warp == kTPvLo) && lane == 0) {
      uint64_t* md = &mma_done[warp == kTQk ? 0 : warp == kTPv ? 1 : 2];
      umma_commit(md);  // arrives once every MMA this thread issued has completed
      mbar_wait(md, 0);
    }
    __syncthreads();
  }
  tc_fence_after();
  if (warp == kTQk) tmem_dealloc(tmem, kTTmemCols);
}

}  // namespace
}  // namespace rgd
