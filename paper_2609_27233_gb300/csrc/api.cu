// C ABI of libumim: host-side argument checks, then the kernels of each part.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace umim {

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);

// cuTensorMapEncodeTiled through the runtime's driver entry point (no -lcuda)
EncodeTiledFn get_encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

// internal entry points (one translation unit per part)
size_t merge_spans_workspace_bytes(int64_t T, int S, int d);
umim_status merge_spans(const void *, int64_t, const int32_t *, int64_t, const int32_t *, int,
                        const umim_merge_weights *, float *, void *, int32_t *, cudaStream_t, int);
size_t build_compressed_workspace_bytes(int B, int S);
umim_status build_compressed(const void *, int64_t, int, const int32_t *, int, int, const int32_t *,
                             const int32_t *, const int32_t *, int, const float *, void *, int64_t, int32_t *,
                             int32_t *, void *, int32_t *, cudaStream_t, int);
size_t kv_rollback_workspace_bytes(int B, int S, int max_pages, int n_layers, int n_kv_heads, int head_dim);
umim_status kv_rollback(const umim_paged_kv *, int32_t *, int32_t, int32_t *, int32_t, const int32_t *,
                        const int32_t *, const int32_t *, int32_t, const void *, const void *, int32_t *, void *,
                        size_t, int32_t *, cudaStream_t, int, const float *, int);
umim_status kv_append(const umim_paged_kv *, int32_t *, int32_t, int32_t *, int32_t, const void *, const void *,
                      const int32_t *, int32_t *, cudaStream_t);
umim_status decode_append_merge(const umim_paged_kv *, int32_t *, int32_t, int32_t *, int32_t, const void *,
                                const void *, const int32_t *, const int32_t *, const int32_t *, int32_t, const void *,
                                const void *, int32_t *, int32_t *, cudaStream_t);
size_t rule_table_bytes(int64_t n_rules);
umim_status rules_build(void *, size_t, const int32_t *, int64_t, int32_t *, cudaStream_t, int);
size_t match_prompts_workspace_bytes(int B, int L);
umim_status match_prompts(const void *, size_t, const int32_t *, int, int, const int32_t *, int32_t *, int32_t *,
                          int32_t *, int32_t *, int32_t *, int32_t *, void *, int32_t *, cudaStream_t, int);
umim_status match_suffix(const void *, size_t, void *, const int32_t *, int, int32_t *, int32_t *, int32_t *,
                         int32_t *, int32_t *, int32_t *, cudaStream_t);
umim_status lookup_surrogates(const float *, int64_t, int, const int32_t *, int, const int32_t *, float *, int32_t *,
                              cudaStream_t, int);
umim_status selftest_bounded_wait(int, uint32_t, const int32_t *, uint64_t *, int32_t *, cudaStream_t);
umim_status selftest_bounds_check(int32_t *, int64_t, int64_t, int32_t *, cudaStream_t);
size_t prefill_attention_workspace_bytes(int B, int T, int Hkv, int D);
umim_status prefill_attention(const void *, const void *, const void *, int, int, int, int, const int32_t *, int,
                              float, void *, void *, int32_t *, cudaStream_t, int);
size_t distill_align_workspace_bytes(int B, int S);
umim_status distill_align(const int32_t *, int32_t, const int32_t *, const int32_t *, const int32_t *, int32_t,
                          int32_t *, int32_t *, int32_t *, int32_t, int32_t *, void *, int32_t *, cudaStream_t);
size_t distill_soft_ce_workspace_bytes(int R_S, int max_pairs);
int distill_soft_ce_vecs(int64_t V);
umim_status distill_soft_ce(const void *, int32_t, const void *, int32_t, int32_t, int64_t, const int32_t *,
                            const int32_t *, int32_t, const int32_t *, float, float *, float *, void *, void *,
                            int32_t *, cudaStream_t, int);
int decode_step_max_batch();
size_t decode_step_workspace_bytes(int B, int Hkv, int D, int num_sms);
umim_status decode_layer_step(const void *, int, const umim_paged_kv *, int, int32_t *, int, int32_t *, int,
                              const void *, const void *, int64_t, const int32_t *, const int32_t *, const int32_t *,
                              int, const void *, const void *, int, int32_t *, float, void *, void *, int32_t *,
                              cudaStream_t, int);
size_t decode_attention_workspace_bytes(int B, int Hq, int Hkv, int D, int num_sms);
umim_status decode_attention(const void *, int, const umim_paged_kv *, int, const int32_t *, int, const int32_t *,
                             int, float, void *, void *, int32_t *, cudaStream_t, int);

namespace {

int current_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return sms;
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

constexpr int64_t kMaxRules = int64_t(1) << 29;

// a rule table buffer: 16-B aligned, a power of two of 16-byte slots, at least 16 of them
bool table_ok(const void *t, size_t bytes) {
  const uint64_t slots = bytes / 16;
  return t && aligned(t, 16) && bytes % 16 == 0 && slots >= 16 && (slots & (slots - 1)) == 0 &&
         slots <= (uint64_t(1) << 31);
}

bool kv_ok(const umim_paged_kv *kv) {
  return kv && kv->base && kv->n_layers > 0 && kv->n_pages > 0 && kv->n_kv_heads > 0 && aligned(kv->base, 16);
}

bool kv_supported(const umim_paged_kv *kv) {
  return kv->page_size == UMIM_PAGE_SIZE && (kv->head_dim == 64 || kv->head_dim == 128) && kv->n_kv_heads <= 64;
}

bool merge_supported(int d, int h) {
  return d > 0 && d % 512 == 0 && d <= 8192 && (h == 1 || h == 2 || h == 4 || h == 8);
}

}  // namespace
}  // namespace umim

using namespace umim;

extern "C" {

const char *umim_status_string(int s) {
  if ((s & 0xff) == UMIM_ERR_BOUNDS) return "UMIM_ERR_BOUNDS";
  switch (s) {
    case UMIM_OK: return "UMIM_OK";
    case UMIM_ERR_INVALID_ARG: return "UMIM_ERR_INVALID_ARG";
    case UMIM_ERR_UNSUPPORTED: return "UMIM_ERR_UNSUPPORTED";
    case UMIM_ERR_CUDA: return "UMIM_ERR_CUDA";
    case UMIM_ERR_TIMEOUT: return "UMIM_ERR_TIMEOUT";
    case UMIM_ERR_WORKSPACE: return "UMIM_ERR_WORKSPACE";
    default: return "UMIM_ERR_UNKNOWN";
  }
}

int umim_version(void) { return 100; }

size_t umim_merge_spans_workspace_size(int64_t n_tokens, int32_t n_spans, int32_t d_model) {
  if (n_tokens < 0 || n_spans < 0 || d_model <= 0) return 0;
  return merge_spans_workspace_bytes(n_tokens, n_spans, d_model);
}

umim_status umim_merge_spans(const void *embeddings, int64_t vocab, const int32_t *token_ids, int64_t n_tokens,
                             const int32_t *span_offsets, int32_t n_spans, const umim_merge_weights *w,
                             float *surrogates, void *workspace, size_t workspace_bytes, int32_t *dev_status,
                             cudaStream_t stream) {
  if (!w || n_spans < 0 || n_tokens < 0 || vocab <= 0) return UMIM_ERR_INVALID_ARG;
  if (!merge_supported(w->d_model, w->n_heads)) return UMIM_ERR_UNSUPPORTED;
  if (n_tokens > (int64_t)n_spans * UMIM_MAX_SPAN_TOKENS || n_tokens > INT32_MAX) return UMIM_ERR_INVALID_ARG;
  if (n_tokens < n_spans) return UMIM_ERR_INVALID_ARG;   // every span has at least one token
  if (n_spans == 0) return UMIM_OK;
  if (!embeddings || !span_offsets || !surrogates || (n_tokens > 0 && !token_ids)) return UMIM_ERR_INVALID_ARG;
  if (!w->w_kv || !w->b_kv || !w->ln_kv_gamma || !w->ln_kv_beta || !w->query || !w->w_o || !w->b_o ||
      !w->ln_o_gamma || !w->ln_o_beta)
    return UMIM_ERR_INVALID_ARG;
  if (!aligned(embeddings, 16) || !aligned(surrogates, 16)) return UMIM_ERR_INVALID_ARG;
  for (const void *p : {w->w_kv, w->b_kv, w->ln_kv_gamma, w->ln_kv_beta, w->query, w->w_o, w->b_o, w->ln_o_gamma,
                        w->ln_o_beta})
    if (!aligned(p, 16)) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < merge_spans_workspace_bytes(n_tokens, n_spans, w->d_model))
    return UMIM_ERR_WORKSPACE;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return merge_spans(embeddings, vocab, token_ids, n_tokens, span_offsets, n_spans, w, surrogates, workspace,
                     dev_status, stream, sms);
}

size_t umim_build_compressed_workspace_size(int32_t batch, int32_t n_spans) {
  if (batch < 0 || n_spans < 0) return 0;
  return build_compressed_workspace_bytes(batch, n_spans);
}

umim_status umim_build_compressed(const void *embeddings, int64_t vocab, int32_t d_model, const int32_t *token_ids,
                                  int32_t batch, int32_t prompt_len, const int32_t *span_offsets,
                                  const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                                  const float *surrogates, void *out_embeds, int64_t out_capacity_rows,
                                  int32_t *position_ids, int32_t *cu_seqlens, void *workspace,
                                  size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream) {
  if (batch < 0 || prompt_len < 0 || n_spans < 0 || vocab <= 0 || out_capacity_rows < 0)
    return UMIM_ERR_INVALID_ARG;
  if (d_model <= 0 || d_model % 8 != 0) return UMIM_ERR_UNSUPPORTED;
  if ((int64_t)batch * prompt_len > INT32_MAX) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!embeddings || !token_ids || !span_offsets || !out_embeds || !position_ids || !cu_seqlens)
    return UMIM_ERR_INVALID_ARG;
  if (n_spans > 0 && (!span_start || !span_len || !surrogates)) return UMIM_ERR_INVALID_ARG;
  if (!aligned(embeddings, 16) || !aligned(out_embeds, 16) || (surrogates && !aligned(surrogates, 16)))
    return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < build_compressed_workspace_bytes(batch, n_spans))
    return UMIM_ERR_WORKSPACE;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return build_compressed(embeddings, vocab, d_model, token_ids, batch, prompt_len, span_offsets, span_start,
                          span_len, n_spans, surrogates, out_embeds, out_capacity_rows, position_ids, cu_seqlens,
                          workspace, dev_status, stream, sms);
}

size_t umim_kv_rollback_workspace_size(int32_t batch, int32_t n_spans, int32_t max_pages, int32_t n_layers,
                                       int32_t n_kv_heads, int32_t head_dim) {
  if (batch < 0 || n_spans < 0 || max_pages < 0 || n_layers <= 0 || n_kv_heads <= 0 ||
      (head_dim != 64 && head_dim != 128))
    return 0;
  return kv_rollback_workspace_bytes(batch, n_spans, max_pages, n_layers, n_kv_heads, head_dim);
}

namespace {
umim_status rollback_checked(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                             int32_t batch, const int32_t *span_offsets, const int32_t *span_start,
                             const int32_t *span_len, int32_t n_spans, const void *surrogate_k,
                             const void *surrogate_v, int32_t *freed_pages, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream,
                             const float *rope_inv_freq, int32_t rotary_dim) {
  if (!kv_ok(kv) || batch < 0 || max_pages < 0 || n_spans < 0) return UMIM_ERR_INVALID_ARG;
  if (!kv_supported(kv)) return UMIM_ERR_UNSUPPORTED;
  if (rope_inv_freq && (rotary_dim <= 0 || rotary_dim % 16 != 0 || rotary_dim > kv->head_dim))
    return UMIM_ERR_INVALID_ARG;
  if ((int64_t)batch * max_pages > INT32_MAX / 16 || batch > 65535) return UMIM_ERR_UNSUPPORTED;
  // work units (sequence x page x layer x K|V x head) are indexed in 32 bits
  if ((int64_t)batch * max_pages * kv->n_layers * 2 * kv->n_kv_heads >= INT32_MAX / 2) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!block_table || !seq_lens || !span_offsets) return UMIM_ERR_INVALID_ARG;
  if (n_spans > 0 && (!span_start || !span_len || !surrogate_k || !surrogate_v)) return UMIM_ERR_INVALID_ARG;
  if (n_spans > 0 && (!aligned(surrogate_k, 16) || !aligned(surrogate_v, 16))) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < kv_rollback_workspace_bytes(batch, n_spans, max_pages, kv->n_layers, kv->n_kv_heads,
                                                    kv->head_dim))
    return UMIM_ERR_WORKSPACE;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return kv_rollback(kv, block_table, max_pages, seq_lens, batch, span_offsets, span_start, span_len, n_spans,
                     surrogate_k, surrogate_v, freed_pages, workspace, workspace_bytes, dev_status, stream, sms,
                     rope_inv_freq, rotary_dim);
}
}  // namespace

umim_status umim_kv_rollback(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                             int32_t batch, const int32_t *span_offsets, const int32_t *span_start,
                             const int32_t *span_len, int32_t n_spans, const void *surrogate_k,
                             const void *surrogate_v, int32_t *freed_pages, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream) {
  return rollback_checked(kv, block_table, max_pages, seq_lens, batch, span_offsets, span_start, span_len, n_spans,
                          surrogate_k, surrogate_v, freed_pages, workspace, workspace_bytes, dev_status, stream,
                          nullptr, 0);
}

umim_status umim_kv_rollback_rope(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages,
                                  int32_t *seq_lens, int32_t batch, const int32_t *span_offsets,
                                  const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                                  const void *surrogate_k, const void *surrogate_v, const float *rope_inv_freq,
                                  int32_t rotary_dim, int32_t *freed_pages, void *workspace, size_t workspace_bytes,
                                  int32_t *dev_status, cudaStream_t stream) {
  if (!rope_inv_freq) return UMIM_ERR_INVALID_ARG;
  return rollback_checked(kv, block_table, max_pages, seq_lens, batch, span_offsets, span_start, span_len, n_spans,
                          surrogate_k, surrogate_v, freed_pages, workspace, workspace_bytes, dev_status, stream,
                          rope_inv_freq, rotary_dim);
}

umim_status umim_kv_append(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                           int32_t batch, const void *new_k, const void *new_v, const int32_t *new_pages,
                           int32_t *dev_status, cudaStream_t stream) {
  if (!kv_ok(kv) || batch < 0 || max_pages < 0) return UMIM_ERR_INVALID_ARG;
  if (!kv_supported(kv)) return UMIM_ERR_UNSUPPORTED;
  if ((int64_t)batch * max_pages > INT32_MAX / 16) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!block_table || !seq_lens || !new_k || !new_v) return UMIM_ERR_INVALID_ARG;
  if (!aligned(new_k, 16) || !aligned(new_v, 16)) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  return kv_append(kv, block_table, max_pages, seq_lens, batch, new_k, new_v, new_pages, dev_status, stream);
}

umim_status umim_decode_append_merge(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages,
                                     int32_t *seq_lens, int32_t batch, const void *new_k, const void *new_v,
                                     const int32_t *new_pages, const int32_t *merge_k, const int32_t *merge_row,
                                     int32_t n_merge_rows, const void *surrogate_k, const void *surrogate_v,
                                     int32_t *released_pages, int32_t *dev_status, cudaStream_t stream) {
  if (!kv_ok(kv) || batch < 0 || max_pages < 0 || n_merge_rows < 0) return UMIM_ERR_INVALID_ARG;
  if (!kv_supported(kv)) return UMIM_ERR_UNSUPPORTED;
  if ((int64_t)batch * max_pages > INT32_MAX / 16) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!block_table || !seq_lens || !new_k || !new_v) return UMIM_ERR_INVALID_ARG;
  if (!aligned(new_k, 16) || !aligned(new_v, 16)) return UMIM_ERR_INVALID_ARG;
  if (merge_k && n_merge_rows > 0 && (!merge_row || !surrogate_k || !surrogate_v)) return UMIM_ERR_INVALID_ARG;
  if (n_merge_rows > 0 && (!aligned(surrogate_k, 16) || !aligned(surrogate_v, 16))) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  return decode_append_merge(kv, block_table, max_pages, seq_lens, batch, new_k, new_v, new_pages, merge_k,
                             merge_row, n_merge_rows, surrogate_k, surrogate_v, released_pages, dev_status, stream);
}

size_t umim_rule_table_bytes(int64_t n_rules) {
  if (n_rules < 0 || n_rules > kMaxRules) return 0;
  return rule_table_bytes(n_rules);
}

umim_status umim_rules_build(void *table, size_t table_bytes, const int32_t *rule_tokens, int64_t n_rules,
                             int32_t *dev_status, cudaStream_t stream) {
  if (n_rules < 0 || n_rules > kMaxRules || !table_ok(table, table_bytes)) return UMIM_ERR_INVALID_ARG;
  if ((uint64_t)table_bytes < 24ull * (uint64_t)n_rules) return UMIM_ERR_WORKSPACE;
  if (n_rules > 0 && (!rule_tokens || !aligned(rule_tokens, 16))) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return rules_build(table, table_bytes, rule_tokens, n_rules, dev_status, stream, sms);
}

size_t umim_match_prompts_workspace_size(int32_t batch, int32_t max_len) {
  if (batch < 0 || max_len < 0) return 0;
  return match_prompts_workspace_bytes(batch, max_len);
}

umim_status umim_match_prompts(const void *table, size_t table_bytes, const int32_t *token_ids, int32_t batch,
                               int32_t max_len, const int32_t *prompt_lens, int32_t *span_offsets,
                               int32_t *span_start, int32_t *span_len, int32_t *span_rule,
                               int32_t *merge_token_ids, int32_t *merge_offsets, void *workspace,
                               size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream) {
  if (!table_ok(table, table_bytes) || batch < 0 || max_len < 0 || !span_offsets) return UMIM_ERR_INVALID_ARG;
  if ((int64_t)batch * max_len >= INT32_MAX) return UMIM_ERR_UNSUPPORTED;
  if ((merge_token_ids == nullptr) != (merge_offsets == nullptr)) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  if (batch == 0) {
    if (cudaMemsetAsync(span_offsets, 0, sizeof(int32_t), stream) != cudaSuccess) return UMIM_ERR_CUDA;
    if (merge_offsets && cudaMemsetAsync(merge_offsets, 0, sizeof(int32_t), stream) != cudaSuccess)
      return UMIM_ERR_CUDA;
    return UMIM_OK;
  }
  if (!token_ids || !span_start || !span_len || !span_rule) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < match_prompts_workspace_bytes(batch, max_len))
    return UMIM_ERR_WORKSPACE;
  return match_prompts(table, table_bytes, token_ids, batch, max_len, prompt_lens, span_offsets, span_start,
                       span_len, span_rule, merge_token_ids, merge_offsets, workspace, dev_status, stream, sms);
}

umim_status umim_match_suffix(const void *table, size_t table_bytes, umim_suffix_state *state,
                              const int32_t *new_tokens, int32_t batch, int32_t *merge_k, int32_t *merge_rule,
                              int32_t *merge_row, int32_t *rows_rule, int32_t *n_merges, int32_t *dev_status,
                              cudaStream_t stream) {
  static_assert(sizeof(umim_suffix_state) == 16, "suffix state is one 16-byte vector");
  if (!table_ok(table, table_bytes) || batch < 0) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  if (batch == 0) {
    if (n_merges && cudaMemsetAsync(n_merges, 0, sizeof(int32_t), stream) != cudaSuccess) return UMIM_ERR_CUDA;
    return UMIM_OK;
  }
  if (!state || !aligned(state, 16) || !new_tokens || !merge_k || !merge_rule || !merge_row)
    return UMIM_ERR_INVALID_ARG;
  return match_suffix(table, table_bytes, state, new_tokens, batch, merge_k, merge_rule, merge_row, rows_rule,
                      n_merges, dev_status, stream);
}

umim_status umim_lookup_surrogates(const float *lut, int64_t n_rules, int32_t d, const int32_t *rule_ids,
                                   int32_t n_max, const int32_t *n_dev, float *out, int32_t *dev_status,
                                   cudaStream_t stream) {
  if (n_rules < 0 || d <= 0 || d % 4 != 0 || n_max < 0) return UMIM_ERR_INVALID_ARG;
  if (n_max == 0) return UMIM_OK;
  if (!lut || !aligned(lut, 16) || !rule_ids || !out || !aligned(out, 16)) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return lookup_surrogates(lut, n_rules, d, rule_ids, n_max, n_dev, out, dev_status, stream, sms);
}

umim_status umim_selftest_bounded_wait(int32_t which, uint32_t limit_us, const int32_t *flags,
                                       uint64_t *elapsed_ns, int32_t *dev_status, cudaStream_t stream) {
  if ((which != 0 && which != 1) || limit_us == 0 || limit_us > 1000000u) return UMIM_ERR_INVALID_ARG;
  if (which == 1 && !flags) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  return selftest_bounded_wait(which, limit_us, flags, elapsed_ns, dev_status, stream);
}

int umim_debug_build(void) { return kDebugChecks ? 1 : 0; }

const char *umim_debug_site_name(int32_t status) {
  static const char *const names[kSiteCount] = {
      "",
      "selftest",
      "rollback_map.block_table",
      "rollback_move.dst_page",
      "rollback_move.src",
      "rollback_move.surrogate",
      "rollback_move.reader_row",
      "append.dst",
      "append.src_row",
      "attention.block_table",
      "attention.piece",
      "decode_step.block_table",
      "decode_step.cache_write",
      "decode_step.partial",
      "merge.pool_stats",
      "merge.gemm_store",
      "merge.pool_span",
      "compaction.token",
      "prefill.kv_row",
      "prefill.out_row",
      "distill.teacher_row",
      "distill.pair",
      "rules.span_slot",
      "rules.span_token",
  };
  const int site = (status >> 8) & 0xffffff;
  return site < kSiteCount ? names[site] : "";
}

umim_status umim_selftest_bounds_check(int32_t *buf, int64_t n, int64_t index, int32_t *dev_status,
                                       cudaStream_t stream) {
  if (!kDebugChecks) return UMIM_ERR_UNSUPPORTED;   // nothing would stop the store: launch nothing
  if (!buf || n <= 0) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  return selftest_bounds_check(buf, n, index, dev_status, stream);
}

size_t umim_prefill_attention_workspace_size(int32_t batch, int32_t n_rows, int32_t n_kv_heads, int32_t head_dim) {
  if (batch < 0 || n_rows < 0 || n_kv_heads <= 0 || (head_dim != 64 && head_dim != 128)) return 0;
  return prefill_attention_workspace_bytes(batch, n_rows, n_kv_heads, head_dim);
}

umim_status umim_prefill_attention(const void *q, const void *k, const void *v, int32_t n_rows, int32_t n_q_heads,
                                   int32_t n_kv_heads, int32_t head_dim, const int32_t *cu_seqlens, int32_t batch,
                                   float scale, void *out, void *workspace, size_t workspace_bytes,
                                   int32_t *dev_status, cudaStream_t stream) {
  if (n_rows < 0 || batch < 0 || n_q_heads <= 0 || n_kv_heads <= 0) return UMIM_ERR_INVALID_ARG;
  if ((head_dim != 64 && head_dim != 128) || n_q_heads % n_kv_heads != 0 || n_q_heads > 65535)
    return UMIM_ERR_UNSUPPORTED;
  if (batch == 0 || n_rows == 0) return UMIM_OK;
  if (!q || !k || !v || !out || !cu_seqlens) return UMIM_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(out, 16)) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < prefill_attention_workspace_bytes(batch, n_rows, n_kv_heads, head_dim))
    return UMIM_ERR_WORKSPACE;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return prefill_attention(q, k, v, n_rows, n_q_heads, n_kv_heads, head_dim, cu_seqlens, batch, scale, out,
                           workspace, dev_status, stream, sms);
}

size_t umim_distill_align_workspace_size(int32_t batch, int32_t n_spans) {
  if (batch < 0 || n_spans < 0) return 0;
  return distill_align_workspace_bytes(batch, n_spans);
}

umim_status umim_distill_align(const int32_t *seq_lens, int32_t batch, const int32_t *span_offsets,
                               const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                               int32_t *pair_offsets, int32_t *teacher_rows, int32_t *student_rows,
                               int32_t capacity, int32_t *student_cu, void *workspace, size_t workspace_bytes,
                               int32_t *dev_status, cudaStream_t stream) {
  if (batch < 0 || n_spans < 0 || capacity < 0 || !pair_offsets) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  if (batch == 0) {
    if (cudaMemsetAsync(pair_offsets, 0, sizeof(int32_t), stream) != cudaSuccess) return UMIM_ERR_CUDA;
    if (student_cu && cudaMemsetAsync(student_cu, 0, sizeof(int32_t), stream) != cudaSuccess) return UMIM_ERR_CUDA;
    return UMIM_OK;
  }
  if (!seq_lens || !span_offsets || (n_spans > 0 && (!span_start || !span_len))) return UMIM_ERR_INVALID_ARG;
  if (capacity > 0 && (!teacher_rows || !student_rows)) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < distill_align_workspace_bytes(batch, n_spans))
    return UMIM_ERR_WORKSPACE;
  return distill_align(seq_lens, batch, span_offsets, span_start, span_len, n_spans, pair_offsets, teacher_rows,
                       student_rows, capacity, student_cu, workspace, dev_status, stream);
}

size_t umim_distill_soft_ce_workspace_size(int32_t n_student_rows, int32_t max_pairs) {
  if (n_student_rows < 0 || max_pairs < 0) return 0;
  return distill_soft_ce_workspace_bytes(n_student_rows, max_pairs);
}

umim_status umim_distill_soft_ce(const void *teacher_logits, int32_t n_teacher_rows, const void *student_logits,
                                 int32_t n_student_rows, int32_t vocab, int64_t ld, const int32_t *teacher_rows,
                                 const int32_t *student_rows, int32_t max_pairs, const int32_t *n_pairs, float eps,
                                 float *loss, float *pair_loss, void *grad, void *workspace,
                                 size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream) {
  if (n_teacher_rows < 0 || n_student_rows < 0 || max_pairs < 0 || vocab < 1 || !loss) return UMIM_ERR_INVALID_ARG;
  if (!(eps >= 0.f) || !std::isfinite(eps)) return UMIM_ERR_INVALID_ARG;
  if (ld % 8 != 0 || ld < ((int64_t)vocab + 7) / 8 * 8) return UMIM_ERR_INVALID_ARG;
  if (distill_soft_ce_vecs(vocab) == 0) return UMIM_ERR_UNSUPPORTED;
  if (n_teacher_rows > 0 && (!teacher_logits || !aligned(teacher_logits, 16))) return UMIM_ERR_INVALID_ARG;
  if (n_student_rows > 0 && (!student_logits || !aligned(student_logits, 16))) return UMIM_ERR_INVALID_ARG;
  if (grad && !aligned(grad, 16)) return UMIM_ERR_INVALID_ARG;
  if (max_pairs > 0 && (!teacher_rows || !student_rows)) return UMIM_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < distill_soft_ce_workspace_bytes(n_student_rows, max_pairs))
    return UMIM_ERR_WORKSPACE;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  return distill_soft_ce(teacher_logits, n_teacher_rows, student_logits, n_student_rows, vocab, ld, teacher_rows,
                         student_rows, max_pairs, n_pairs, eps, loss, pair_loss, grad, workspace, dev_status,
                         stream, sms);
}

size_t umim_decode_attention_workspace_size(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads,
                                            int32_t head_dim) {
  if (batch < 0 || n_q_heads <= 0 || n_kv_heads <= 0 || (head_dim != 64 && head_dim != 128)) return 0;
  int sms = current_sms();
  if (sms <= 0) sms = 256;   // no device yet: size for the largest grid this library launches
  return decode_attention_workspace_bytes(batch, n_q_heads, n_kv_heads, head_dim, sms);
}

umim_status umim_decode_attention(const void *q, int32_t n_q_heads, const umim_paged_kv *kv, int32_t layer,
                                  const int32_t *block_table, int32_t max_pages, const int32_t *seq_lens,
                                  int32_t batch, float scale, void *out, void *workspace, size_t workspace_bytes,
                                  int32_t *dev_status, cudaStream_t stream) {
  if (!kv_ok(kv) || batch < 0 || max_pages < 0 || n_q_heads <= 0) return UMIM_ERR_INVALID_ARG;
  if (!kv_supported(kv)) return UMIM_ERR_UNSUPPORTED;
  if (n_q_heads % kv->n_kv_heads != 0 || n_q_heads / kv->n_kv_heads > 16) return UMIM_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= kv->n_layers) return UMIM_ERR_INVALID_ARG;
  if ((int64_t)batch * kv->n_kv_heads > (int64_t)1 << 24) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!q || !block_table || !seq_lens || !out) return UMIM_ERR_INVALID_ARG;
  if (!aligned(q, 4) || !aligned(out, 2)) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < decode_attention_workspace_bytes(batch, n_q_heads, kv->n_kv_heads, kv->head_dim, sms))
    return UMIM_ERR_WORKSPACE;
  if (!(scale > 0.f)) scale = 1.0f / sqrtf((float)kv->head_dim);
  int32_t *status = dev_status;
  return decode_attention(q, n_q_heads, kv, layer, block_table, max_pages, seq_lens, batch, scale, out, workspace,
                          status, stream, sms);
}

size_t umim_decode_layer_step_workspace_size(int32_t batch, int32_t n_kv_heads, int32_t head_dim) {
  if (batch < 0 || n_kv_heads <= 0 || (head_dim != 64 && head_dim != 128)) return 0;
  int sms = current_sms();
  if (sms <= 0) sms = 256;   // no device yet: size for the largest grid this library launches
  return decode_step_workspace_bytes(batch, n_kv_heads, head_dim, sms);
}

umim_status umim_decode_layer_step(const void *q, int32_t n_q_heads, const umim_paged_kv *kv, int32_t layer,
                                   int32_t *block_table, int32_t max_pages, int32_t *seq_lens, int32_t batch,
                                   const void *new_k, const void *new_v, int64_t new_row_stride,
                                   const int32_t *new_pages, const int32_t *merge_k, const int32_t *merge_row,
                                   int32_t n_merge_rows, const void *surrogate_k, const void *surrogate_v,
                                   int32_t commit, int32_t *released_pages, float scale, void *out, void *workspace,
                                   size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream) {
  if (!kv_ok(kv) || batch < 0 || max_pages < 0 || n_q_heads <= 0 || n_merge_rows < 0 || new_row_stride < 0)
    return UMIM_ERR_INVALID_ARG;
  if (!kv_supported(kv)) return UMIM_ERR_UNSUPPORTED;
  if (n_q_heads % kv->n_kv_heads != 0 || n_q_heads / kv->n_kv_heads > 16) return UMIM_ERR_UNSUPPORTED;
  if (batch > decode_step_max_batch() || (int64_t)batch * max_pages > INT32_MAX / 16) return UMIM_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= kv->n_layers) return UMIM_ERR_INVALID_ARG;
  if (batch == 0) return UMIM_OK;
  const int64_t row = (int64_t)kv->n_kv_heads * kv->head_dim;
  if (new_row_stride == 0) new_row_stride = row;
  if (new_row_stride < row || new_row_stride % 8 != 0) return UMIM_ERR_INVALID_ARG;
  if (!q || !block_table || !seq_lens || !out || !new_k || !new_v) return UMIM_ERR_INVALID_ARG;
  if (!aligned(q, 4) || !aligned(out, 4) || !aligned(new_k, 16) || !aligned(new_v, 16)) return UMIM_ERR_INVALID_ARG;
  if (merge_k && n_merge_rows > 0 && (!merge_row || !surrogate_k || !surrogate_v)) return UMIM_ERR_INVALID_ARG;
  if (n_merge_rows > 0 && (!aligned(surrogate_k, 16) || !aligned(surrogate_v, 16))) return UMIM_ERR_INVALID_ARG;
  const DeviceScope scope(stream);
  const int sms = scope.sms();
  if (!workspace || !aligned(workspace, 256) ||
      workspace_bytes < decode_step_workspace_bytes(batch, kv->n_kv_heads, kv->head_dim, sms))
    return UMIM_ERR_WORKSPACE;
  if (!(scale > 0.f)) scale = 1.0f / sqrtf((float)kv->head_dim);
  return decode_layer_step(q, n_q_heads, kv, layer, block_table, max_pages, seq_lens, batch, new_k, new_v,
                           new_row_stride, new_pages, merge_k, merge_row, n_merge_rows, surrogate_k, surrogate_v,
                           commit != 0, released_pages, scale, out, workspace, dev_status, stream, sms);
}

}  // extern "C"
