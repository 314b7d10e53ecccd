/*
 * rgd.h -- C ABI of the refusal-gated decode step on GB300 (sm_103a).
 *
 * Refusal-gated decoding (arxiv 2607.20791) runs, for every prompt, one greedy
 * "probe" row and N high-temperature sample rows.  All rows of a prompt attend
 * to the prompt's KV cache, which is computed once and reused (Sec. 3), plus
 * their own generated-suffix KV.  The greedy probe is checked token by token
 * against a set P of refusal prefixes (the compatibility predicate C, Sec. 3;
 * matched on token prefixes, a detection needing at least two tokens, App. D);
 * the hard gate of Alg. 1 then either keeps the greedy refusal or discards the
 * probe and keeps the high-temperature samples.
 *
 * This library implements one decode step of that loop as CUDA kernels:
 *   rgd_prefix_decode_attn  shared-prefix split-KV decode attention,
 *   rgd_sample_head         greedy argmax / temperature + min-p + Philox sample,
 *   rgd_probe_gate          per-token refusal-prefix gate on a token trie,
 *   rgd_sample_head_gated   the two above in one kernel,
 *   rgd_decode_step         attention, then the gated head: one whole step,
 *   rgd_soft_gate           its soft variant (the appendix ablation, Alg. 2),
 *   rgd_residual_precheck   the residual-stream classifier that lets a prompt
 *                           skip the probe (App. A), once per prompt.
 *
 * Conventions for every entry point
 *   - Tensor pointers are DEVICE pointers owned by the caller unless a comment
 *     says "host".  The library never frees them.  bf16 values are passed as
 *     their 16-bit patterns (rgd_bf16).  All tensors are dense, row-major, with
 *     the shapes given, and 16-byte aligned base addresses.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = the legacy
 *     default stream) and use the device that is current on the calling thread.
 *   - The return value is a host status: RGD_OK, or an RGD_ERR_* code when the
 *     arguments are rejected (nothing is launched) or a launch fails;
 *     rgd_last_error_string() then describes the error (per thread).
 *   - Errors found on the device (an out-of-range page id, an invalid
 *     temperature, a wait that timed out) never trap: the kernel ORs an
 *     RGD_DEV_* bit into *dev_status (a caller-owned device int32, may be NULL)
 *     and skips the offending work.  Read it after synchronising.
 */
#ifndef RGD_H
#define RGD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* host status codes */
#define RGD_OK 0
#define RGD_ERR_INVALID_ARG 1
#define RGD_ERR_CUDA 2
#define RGD_ERR_UNSUPPORTED 3

/* device status bits (ORed into *dev_status) */
#define RGD_DEV_BAD_PAGE 1      /* block-table entry outside [0, num_pages): read as zeros */
#define RGD_DEV_BAD_TOKEN 2     /* negative probe token that is not the stop token: skipped */
#define RGD_DEV_WAIT_TIMEOUT 4  /* a bounded wait on a copy gave up; outputs of that block are missing */
#define RGD_DEV_BAD_PARAM 8     /* temperature < 0 or not finite, min_p outside [0, 1], or non-finite logits max */

/* logits element types */
#define RGD_F32 0
#define RGD_BF16 1

/* gate decisions (Sec. 3 / Alg. 1 outcomes) */
#define RGD_PENDING 0
#define RGD_REFUSAL 1      /* the greedy probe stays refusal-compatible: return the greedy refusal */
#define RGD_NON_REFUSAL 2  /* the probe became incompatible: discard it, keep the samples */

typedef uint16_t rgd_bf16;
typedef void* rgd_stream_t;

/* Description of the last error on this thread ("" if none). */
const char* rgd_last_error_string(void);
/* Library version string. */
const char* rgd_version(void);

/* ------------------------------------------------------------------------ */
/* Shared-prefix decode attention (Sec. 3: prompt KV reused by the probe and   */
/* the sampling stage; here read once per prompt group and kv head)            */
/* ------------------------------------------------------------------------ */

/* Shape of one attention call.  R = num_groups * rows_per_group rows; row
 * g*rows_per_group is the probe of group g, the next rows_per_group-1 rows are
 * its sample rows.  Query head j uses kv head j / (num_q_heads/num_kv_heads). */
typedef struct {
  int32_t num_groups;        /* G >= 1                                          */
  int32_t rows_per_group;    /* 1 + N >= 1                                      */
  int32_t num_q_heads;       /* Hq, a multiple of num_kv_heads                  */
  int32_t num_kv_heads;      /* Hkv >= 1                                        */
  int32_t head_dim;          /* D: 64 or 128                                    */
  int32_t page_size;         /* tokens per KV page: 16                          */
  int32_t num_pages;         /* pages in each of the K and V pools              */
  int32_t max_prompt_pages;  /* columns of prompt_block_table (>= 1)            */
  int32_t max_suffix_pages;  /* columns of suffix_block_table (>= 1)            */
  int32_t num_ctas;          /* persistent blocks (<= 65535); 0 = one per SM     */
  int32_t reserved;          /* must be 0                                       */
} rgd_attn_shape;

/* Sets how long the attention kernel's blocks wait for one another (a split
 * job's merger for its other pieces) and for their own copies and MMAs before
 * giving up with RGD_DEV_WAIT_TIMEOUT, for every later call on any thread; 0
 * restores the default of 2 s.  The kernel never traps: a wait that gives up
 * stops that block's work, drains its copies in flight and returns.  A short
 * limit serves tests of that path; in service a limit must stay far above a
 * call's run time. */
int rgd_set_wait_limit_ns(uint64_t limit_ns);

/* Bytes of device workspace rgd_prefix_decode_attn needs for this shape (it
 * depends on the current device's SM count when num_ctas is 0). */
size_t rgd_prefix_decode_attn_workspace_size(const rgd_attn_shape* shape);

/* Decode attention of every active row over [prompt KV of its group | its own
 * suffix KV] (the concatenation; no causal mask; no rotary embedding):
 *   out[r, j, :] = softmax(softmax_scale * K q[r, j]) V,
 *   lse[r, j]    = ln sum exp(softmax_scale * K q[r, j])   (natural log).
 * Every prompt KV page of a group is read once and attended by all
 * rows_per_group * Hq/Hkv queries of that group and kv head; a row's suffix
 * pages are attended by that row's queries.  The pages of all (group, kv head)
 * jobs are divided evenly over num_ctas persistent blocks; a job split across
 * blocks is merged from its partial results by log-sum-exp.
 *
 *   q                  bf16 [R, Hq, D]
 *   k_pages, v_pages   bf16 [num_pages, Hkv, page_size, D]
 *   prompt_block_table int32 [G, max_prompt_pages]: page ids of prompt tokens
 *                      (token t in page table[t / page_size], slot t % page_size)
 *   prompt_len         int32 [G], 0 <= prompt_len <= max_prompt_pages*page_size
 *   suffix_block_table int32 [R, max_suffix_pages]
 *   suffix_len         int32 [R], 0 <= suffix_len <= max_suffix_pages*page_size
 *   row_active         uint8 [R] or NULL (all active); inactive rows read no KV
 *                      and their out/lse are left untouched
 *   softmax_scale      > 0 (1/sqrt(D) for standard attention)
 *   out                bf16 [R, Hq, D]; lse float [R, Hq] or NULL
 *   workspace          device memory of rgd_prefix_decode_attn_workspace_size()
 *                      bytes, 256-byte aligned, zero-filled before its first
 *                      use.  It starts with an area of max(J, 8192) int32
 *                      counters, J = num_groups * num_kv_heads (one per (group,
 *                      kv head) job), which every call leaves at zero again
 *                      unless it reports RGD_DEV_WAIT_TIMEOUT (then zero-fill it
 *                      before reuse); the rest is scratch that a call writes
 *                      before reading.  So one workspace, sized for the largest
 *                      shape, may serve calls of any shapes with J <= 8192;
 *                      a call with J > 8192 moves the scratch, so zero-fill the
 *                      workspace whenever the shape changes across it.  Calls
 *                      that share a workspace must not overlap in time.
 * One kernel runs on `stream`.  A job split across blocks is merged by the
 * block holding its first page, which waits (bounded) for the job's other
 * pieces; those are the first pieces of later blocks and wait on no other
 * block, so the wait ends as long as blocks start in index order (num_ctas
 * above the number of blocks the device holds at once relies on that).
 * A group with prompt_len 0 and a row with suffix_len 0 are valid; a row with
 * neither gets out = 0, lse = -inf.  Page ids outside [0, num_pages) read as
 * zeros and set RGD_DEV_BAD_PAGE.  Lengths beyond the table are rejected on the
 * device (RGD_DEV_BAD_PAGE) because the host does not read device lengths. */
int rgd_prefix_decode_attn(const rgd_attn_shape* shape, const rgd_bf16* q,
                           const rgd_bf16* k_pages, const rgd_bf16* v_pages,
                           const int32_t* prompt_block_table, const int32_t* prompt_len,
                           const int32_t* suffix_block_table, const int32_t* suffix_len,
                           const uint8_t* row_active, float softmax_scale, rgd_bf16* out,
                           float* lse, void* workspace, size_t workspace_bytes,
                           int32_t* dev_status, rgd_stream_t stream);

/* Allocation-free form of rgd_prefix_decode_attn (the paper has no counterpart;
 * this is a deployment convenience).  Same arguments and results, minus the
 * workspace: the split partials live in one fixed 8 MiB device
 * array inside the library (one per device, held by every process that loads the
 * library until it exits).  It is for callers that cannot call cudaMalloc: for
 * example a serving engine whose KV-cache manager has already reserved the free
 * device memory (a new allocation would fail or break its memory accounting),
 * or a latency-critical decode loop where cudaMalloc / cudaFree would
 * synchronise the device.  The caller still passes every input and output.
 *   - Shapes whose workspace (rgd_prefix_decode_attn_workspace_size) exceeds
 *     8 MiB, or with more than 8192 (group, kv head) jobs, are rejected with
 *     RGD_ERR_UNSUPPORTED.
 *   - The first call on a device looks up the array's device address (once per
 *     device, with that device current); make that first call before any stream
 *     capture.
 *   - Nothing is allocated or cleared: the array starts zeroed when the library
 *     is loaded; its first 32 KiB hold the job counters of every call, whatever
 *     the shape, and every call leaves the counters of its jobs at zero, unless
 *     it reports RGD_DEV_WAIT_TIMEOUT (after which this entry point must not be
 *     used again in the process).  Every call shares the one array, so calls
 *     that overlap on the GPU (other streams, other threads) race: serialise
 *     them. */
int rgd_prefix_decode_attn_noalloc(const rgd_attn_shape* shape, const rgd_bf16* q,
                                   const rgd_bf16* k_pages, const rgd_bf16* v_pages,
                                   const int32_t* prompt_block_table, const int32_t* prompt_len,
                                   const int32_t* suffix_block_table, const int32_t* suffix_len,
                                   const uint8_t* row_active, float softmax_scale, rgd_bf16* out,
                                   float* lse, int32_t* dev_status, rgd_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Sample head: G_M's greedy token and S_{T,theta}'s truncated sample          */
/* (Sec. 3, Alg. 1; truncation = min-p, Sec. 1)                                */
/* ------------------------------------------------------------------------ */

/* For every active row r of logits [rows, vocab] (RGD_F32 or RGD_BF16):
 *   greedy rows (is_probe[r] != 0 or temperature[r] == 0):
 *     token = argmax, lowest index on ties; kept_count = 1.
 *   sample rows: l_max = max logit; cutoff c = fl32(l_max + fl32(T ln p_min))
 *     (T ln p_min evaluated in double, rounded once to float; p_min = 0 keeps
 *     everything); kept set K = {i : l_i >= c} (this is {p_i >= p_min p_max}
 *     for p = softmax(l/T)); w_i = exp((l_i - l_max)/T); u = Philox4x32-10
 *     uniform with key = seed[r] (low word first) and counter = (step low,
 *     step high, 0, 0): u = (word0 >> 8) * 2^-24; token = the smallest i in K
 *     with sum_{j in K, j <= i} w_j > u * sum_K w.
 *   token_out int32 [rows] (-1 for inactive rows and rejected parameters);
 *   kept_count int32 [rows] or NULL: |K| (0 for inactive rows);
 *   kept_mask uint8 [rows, vocab] or NULL: 1 where i in K (sample rows only;
 *     rows that are greedy or inactive are not written).
 * is_probe may be NULL (no probe rows); row_active may be NULL (all active).
 * vocab must satisfy vocab * element size <= 8 * 200 KiB. */
int rgd_sample_head(int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                    const uint8_t* is_probe, const float* temperature, const float* min_p,
                    const uint64_t* seed, uint64_t step, const uint8_t* row_active,
                    int32_t* token_out, int32_t* kept_count, uint8_t* kept_mask,
                    int32_t* dev_status, rgd_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Refusal-prefix gate (compatibility predicate C, Sec. 3; hard gate, Alg. 1)  */
/* ------------------------------------------------------------------------ */

/* Token trie of the refusal-prefix set P, built on the host and uploaded to the
 * current device.  Library-owned; release with rgd_trie_destroy. */
typedef struct rgd_trie rgd_trie;

/* tokens (host) int32 [offsets[n_seq]]: the sequences back to back, each token
 * >= 0; offsets (host) int64 [n_seq + 1], offsets[0] = 0, strictly increasing
 * (every sequence non-empty).  Duplicates and sequences that are prefixes of
 * others are allowed.  min_confirm >= 1 is the minimum length of a refusal
 * prefix whose full match confirms a refusal (2 in the paper, App. D).
 * n_seq = 0 gives the empty set (every probe is incompatible). */
int rgd_trie_create(const int32_t* tokens, const int64_t* offsets, int32_t n_seq,
                    int32_t min_confirm, rgd_trie** out);
int rgd_trie_destroy(rgd_trie* trie);
/* Node and edge counts of a trie (root included). */
int rgd_trie_info(const rgd_trie* trie, int32_t* num_nodes, int32_t* num_edges);

/* Per-group gate state, in device memory owned by the caller. */
typedef struct {
  int32_t node;           /* trie node of the probe q (root = 0)                    */
  int32_t length;         /* |q|: probe tokens appended (stop token excluded)        */
  int32_t steps;          /* probe tokens consumed (stop token included)             */
  int32_t decisive_step;  /* 0-based index of the token that decided; -1 if pending  */
  uint8_t decision;       /* RGD_PENDING / RGD_REFUSAL / RGD_NON_REFUSAL             */
  uint8_t confirmed;      /* some refusal prefix of length >= min_confirm prefixes q */
  uint8_t done;           /* the probe has ended (stop token, length cap, discarded) */
  uint8_t reserved;       /* 0 between calls (rgd_sample_head_gated counts rows here) */
} rgd_gate_state;

/* Reset `groups` states to the empty probe (node 0, pending). */
int rgd_gate_state_init(rgd_gate_state* state, int32_t groups, rgd_stream_t stream);

/* Feed n_tokens greedy probe tokens per group to the hard gate.  Token k of
 * group g is probe_tokens[g * token_stride + k] (token_stride >= n_tokens; use
 * the sample head's token_out with token_stride = rows_per_group and n_tokens =
 * 1 to gate the probe row of every group).  For each token of a group whose
 * probe has not ended:
 *   - the stop token (eos_token >= 0) ends the probe: REFUSAL if q is
 *     compatible (q non-empty, or P non-empty), else NON_REFUSAL;
 *   - otherwise q <- q || y; if q is not compatible: NON_REFUSAL, the probe
 *     ends; if a refusal prefix of length >= min_confirm is now a prefix of q:
 *     confirmed, REFUSAL (the probe continues to produce its text); if |q|
 *     reaches max_len: the probe ends, REFUSAL if still pending.
 * Then row_active [groups*rows_per_group] (updated in place, may be NULL):
 * the probe row is cleared once the probe has ended; the sample rows of a group
 * are cleared once its decision is REFUSAL.  Negative tokens other than the
 * stop token are skipped and set RGD_DEV_BAD_TOKEN. */
int rgd_probe_gate(const rgd_trie* trie, int32_t groups, int32_t rows_per_group,
                   const int32_t* probe_tokens, int32_t n_tokens, int64_t token_stride,
                   int32_t eos_token, int32_t max_len, rgd_gate_state* state,
                   uint8_t* row_active, int32_t* dev_status, rgd_stream_t stream);

/* The sample head and the hard gate of one decode step in one kernel (Alg. 1:
 * the greedy step G_M and the sample rows' S_{T,theta} draw, then the probe
 * token through the compatibility gate).  Same results as rgd_sample_head
 * (without kept_mask) followed by
 *   rgd_probe_gate(trie, rows / rows_per_group, rows_per_group, token_out, 1,
 *                  rows_per_group, eos_token, max_len, state, row_active, ...):
 * every active row draws its token first, and only then are the rows of a
 * group masked by its gate outcome (the gate of group g runs once all
 * rows_per_group rows of the group have their tokens).  Rows g*rows_per_group
 * .. +rows_per_group-1 form group g; row g*rows_per_group is its probe (pass
 * is_probe with those rows set, or temperature 0 there, for a greedy probe).
 *   row_active   uint8 [rows] or NULL: read as by rgd_sample_head, then
 *                updated in place by the gate
 *   state        device rgd_gate_state [rows / rows_per_group], 4-byte
 *                aligned; its `reserved` byte must be 0 between calls (the
 *                kernel counts a group's finished rows there during the call
 *                and leaves it at 0; rgd_gate_state_init sets it)
 *   rows_per_group in [1, 255], dividing rows; max_len >= 1; trie non-NULL.
 * One kernel on `stream`, launched as a programmatic dependent of the previous
 * kernel on the stream (it is scheduled while that kernel finishes and waits
 * for it before reading any input). */
int rgd_sample_head_gated(int32_t rows, int32_t vocab, int32_t dtype, const void* logits,
                          const uint8_t* is_probe, const float* temperature, const float* min_p,
                          const uint64_t* seed, uint64_t step, uint8_t* row_active, int32_t* token_out,
                          int32_t* kept_count, const rgd_trie* trie, int32_t rows_per_group,
                          int32_t eos_token, int32_t max_len, rgd_gate_state* state, int32_t* dev_status,
                          rgd_stream_t stream);

/* One whole decode step of the gated loop: rgd_prefix_decode_attn over the
 * step's rows, then rgd_sample_head_gated over the step's logits (two kernels
 * on `stream`; the head's blocks are scheduled while the attention finishes).
 * The logits are the caller's: the model between the attention output and the
 * next-token logits (projections, MLP, LM head) is not part of this library.
 * Arguments are those of the two calls, with rows = num_groups *
 * rows_per_group and one row_active shared by both (the attention reads it,
 * the gate updates it); out and lse receive the attention output.  The first
 * error stops the step (nothing after it is launched). */
int rgd_decode_step(const rgd_attn_shape* shape, const rgd_bf16* q, const rgd_bf16* k_pages,
                    const rgd_bf16* v_pages, const int32_t* prompt_block_table, const int32_t* prompt_len,
                    const int32_t* suffix_block_table, const int32_t* suffix_len, float softmax_scale,
                    rgd_bf16* out, float* lse, void* workspace, size_t workspace_bytes, int32_t vocab,
                    int32_t dtype, const void* logits, const uint8_t* is_probe, const float* temperature,
                    const float* min_p, const uint64_t* seed, uint64_t step, uint8_t* row_active,
                    int32_t* token_out, int32_t* kept_count, const rgd_trie* trie, int32_t eos_token,
                    int32_t max_len, rgd_gate_state* state, int32_t* dev_status, rgd_stream_t stream);

/* Soft compatibility gate (the appendix ablation's Alg. 2): one probe step per
 * group from the probe row's logits.  With y the greedy token (argmax, lowest
 * index on ties): after the first c probe steps, or when y is the stop token,
 * or when q || y stays refusal-compatible, this is the hard gate's step with
 * y.  Otherwise the top_k tokens of softmax(logits) (larger logit first, lower
 * index first on ties) that keep q compatible -- the trie children of q's node,
 * and the stop token, which does not change q -- form A_ref with mass m (their
 * softmax probabilities summed); when A_ref is non-empty and m >= rho the most
 * probable of them, a*, is appended instead of y (the caller feeds it back as
 * the probe's token), else the probe is discarded: NON_REFUSAL at this step.
 *   probe_logits   device [groups rows of row_stride elements]: group g's probe
 *                  logits at probe_logits + g * row_stride (RGD_F32 / RGD_BF16);
 *                  use the step's logits with row_stride = rows_per_group * vocab
 *   token_out      device int32 [groups]: the token appended this step (y or
 *                  a*), -1 when none (probe discarded or already ended)
 *   mass_out       device float [groups] or NULL: m when the soft branch ran,
 *                  else -1
 * State and row_active as for rgd_probe_gate.  m is accumulated in fp32 with
 * e^x taken as 2^(x log2 e) by the SFU (the decision can differ from exact
 * arithmetic only when m is within ~1e-5 relative of rho).  dev_status (may
 * be NULL) gets RGD_DEV_WAIT_TIMEOUT when a bounded wait on a copy of the
 * logits gave up; that step's outputs are then not valid.
 * RGD_ERR_UNSUPPORTED when a trie node has more than 2047 children.  One
 * kernel on `stream`: a cluster of 6 blocks per group, each block reading a
 * sixth of the probe row. */
int rgd_soft_gate(const rgd_trie* trie, int32_t groups, int32_t rows_per_group, int32_t vocab, int32_t dtype,
                  const void* probe_logits, int64_t row_stride, int32_t top_k, float rho, int32_t c,
                  int32_t eos_token, int32_t max_len, rgd_gate_state* state, uint8_t* row_active,
                  int32_t* token_out, float* mass_out, int32_t* dev_status, rgd_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Residual-stream precheck (App. A)                                          */
/* ------------------------------------------------------------------------ */

/* Logistic readout of each group's last-prompt-token activation, run once
 * before the probe's first token:
 *   z_g = sum_i w[i] * h[g, i] + bias,  p_g = 1 / (1 + exp(-z_g)),
 * and a group with p_g <= theta skips the greedy probe (App. A: the prompt
 * decodes directly at high temperature).  For such a group whose state is
 * still the fresh empty probe (pending, no token consumed), the state becomes
 * decision RGD_NON_REFUSAL, done = 1, decisive_step -1 (decided before any
 * probe token), and its probe row (row g * rows_per_group) is cleared in
 * row_active; the sample rows stay on.  Other groups are left unchanged.
 *   h           device, [groups, d], dtype RGD_F32 or RGD_BF16, row-major
 *   w           device float [d]; bias, theta in [0, 1] by value
 *   prob_out    device float [groups] (p_g) or NULL
 *   state       device rgd_gate_state [groups]; row_active device
 *               uint8 [groups * rows_per_group] or NULL
 * z is accumulated in fp32 (the decision can differ from exact arithmetic
 * only when z is within the fp32 rounding of its sum from the threshold's
 * logit).  One kernel on `stream`, one block per group. */
int rgd_residual_precheck(int32_t groups, int32_t d, int32_t dtype, const void* h, const float* w, float bias,
                          float theta, int32_t rows_per_group, float* prob_out, rgd_gate_state* state,
                          uint8_t* row_active, int32_t* dev_status, rgd_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RGD_H */
