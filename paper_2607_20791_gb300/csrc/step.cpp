// One decode step of the gated loop (Alg. 1) through the library's own calls:
// the shared-prefix attention, then the sample head with the hard gate fused in.
#include "common.h"

extern "C" int rgd_decode_step(const rgd_attn_shape* shape, const rgd_bf16* q, const rgd_bf16* k_pages,
                               const rgd_bf16* v_pages, const int32_t* prompt_block_table,
                               const int32_t* prompt_len, const int32_t* suffix_block_table,
                               const int32_t* suffix_len, float softmax_scale, rgd_bf16* out, float* lse,
                               void* workspace, size_t workspace_bytes, int32_t vocab, int32_t dtype,
                               const void* logits, const uint8_t* is_probe, const float* temperature,
                               const float* min_p, const uint64_t* seed, uint64_t step, uint8_t* row_active,
                               int32_t* token_out, int32_t* kept_count, const rgd_trie* trie, int32_t eos_token,
                               int32_t max_len, rgd_gate_state* state, int32_t* dev_status, rgd_stream_t stream) {
  rgd::clear_error();
  RGD_CHECK_ARG(shape != nullptr, "rgd_decode_step: shape is NULL");
  const int64_t rows = (int64_t)shape->num_groups * shape->rows_per_group;
  RGD_CHECK_ARG(rows >= 0 && rows <= 0x7fffffff, "rgd_decode_step: too many rows");
  // the head's arguments first, so that a rejected step launches nothing
  if (int rc = rgd::check_gated_head("rgd_decode_step", (int32_t)rows, vocab, dtype, logits, temperature, min_p,
                                     seed, token_out, trie, shape->rows_per_group, max_len, state))
    return rc;
  if (int rc = rgd_prefix_decode_attn(shape, q, k_pages, v_pages, prompt_block_table, prompt_len,
                                      suffix_block_table, suffix_len, row_active, softmax_scale, out, lse,
                                      workspace, workspace_bytes, dev_status, stream))
    return rc;
  return rgd_sample_head_gated((int32_t)rows, vocab, dtype, logits, is_probe, temperature, min_p, seed, step,
                               row_active, token_out, kept_count, trie, shape->rows_per_group, eos_token,
                               max_len, state, dev_status, stream);
}
