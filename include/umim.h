/*
 * umim.h - C ABI of libumim, a GB300 (sm_103a) implementation of the decode
 * step over a merged context of UMIM (arXiv 2609.27233, "Distilling
 * Sequential Computation in Transformer Language Models").
 *
 * The step has three parts, each a call below:
 *   umim_merge_spans       merge module M_phi: span of static token
 *                          embeddings -> one surrogate embedding
 *                          (Sec. 3.2 Eq. 1, App. C.1)
 *   umim_kv_rollback       replace each span's stored KV entries by one
 *                          surrogate entry and compact the paged cache
 *                          (App. C.6, App. E "Decoding-Time Merging and
 *                          KV-Cache Update", Fig. 2)
 *   umim_decode_attention  grouped-query decode attention over the shorter,
 *                          compacted paged cache (App. I.1)
 * and one call for the prompt side:
 *   umim_build_compressed  packed compressed prompt embeddings with
 *                          contiguous positions (App. C.5, App. E "Prompt
 *                          Merging", App. J.4)
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Pointers named *device* point to GPU memory of the current device; the
 *    caller allocates and owns every buffer, including the workspace.  The
 *    library never allocates GPU memory.
 *  - Each call runs on the device of `stream` and restores the caller's
 *    current device before returning.  While `stream` is being captured
 *    into a CUDA graph its device cannot be queried: the current device must
 *    then be the stream's device.
 *  - Every call is asynchronous on `stream`.  The returned umim_status only
 *    reports what the host can check (null pointers, unsupported shapes, a
 *    workspace that is too small, a failed launch).  Checks that need device
 *    data (span lists, token ids, block-table entries) and bounded waits run
 *    on the GPU and record the first failure in `*dev_status` (a device
 *    int32 the caller zeroes; NULL means "use a word inside the workspace and
 *    do not report").  Read it after synchronising the stream.
 *  - bf16 means IEEE bfloat16 (raw 16-bit patterns); fp32 is IEEE binary32.
 *  - Paged KV cache: pages of UMIM_PAGE_SIZE (16) entries; one entry holds
 *    K and V of every KV head of one token position for one layer.
 *    Layout of the pool, bf16, row-major:
 *        [n_layers][n_pages][2 (K, V)][n_kv_heads][16][head_dim]
 *    so one (layer, page, K|V, head) tile of 16 x head_dim values is
 *    contiguous.  A block table row lists, for logical page p of a sequence,
 *    the physical page id (or -1 for none).  Entry t of a sequence lives in
 *    page block_table[t / 16], slot t % 16.
 *  - Supported: head_dim 64 or 128, page size 16, 1 <= n_q_heads/n_kv_heads
 *    <= 16, d_model a multiple of 512 (<= 8192), n_heads in {1, 2, 4, 8},
 *    merge spans of 1..4 tokens.
 *    Anything else returns UMIM_ERR_UNSUPPORTED.
 */
#ifndef UMIM_H_
#define UMIM_H_

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h> /* cudaStream_t */

#ifdef __cplusplus
extern "C" {
#endif

#define UMIM_PAGE_SIZE 16
#define UMIM_MAX_SPAN_TOKENS 4

typedef enum umim_status {
  UMIM_OK = 0,
  UMIM_ERR_INVALID_ARG = 1, /* bad pointer, size, span list, id or page */
  UMIM_ERR_UNSUPPORTED = 2, /* shape outside the supported set above     */
  UMIM_ERR_CUDA = 3,        /* a CUDA runtime / driver call failed       */
  UMIM_ERR_TIMEOUT = 4,     /* a bounded device-side wait gave up        */
  UMIM_ERR_WORKSPACE = 5,   /* workspace pointer or size insufficient    */
  UMIM_ERR_BOUNDS = 6       /* debug build only: an access-site check    */
                            /* failed; the word holds 6 | site << 8      */
} umim_status;

/* Human-readable name of a status code (static string); a debug build's
 * UMIM_ERR_BOUNDS | site << 8 reads as "UMIM_ERR_BOUNDS". */
const char *umim_status_string(int status);

/* Library version as 10000*major + 100*minor + patch. */
int umim_version(void);

/* Merge-module parameters phi (App. C.3: |phi| = 2 d^2 + 7 d), all bf16
 * device arrays, Linear weights stored W[out][in] row-major. */
typedef struct umim_merge_weights {
  const void *w_kv;        /* [d][d]   W^{kv}                              */
  const void *b_kv;        /* [d]      b^{kv}                              */
  const void *ln_kv_gamma; /* [d]      LN_kv scale                         */
  const void *ln_kv_beta;  /* [d]      LN_kv shift                         */
  const void *query;       /* [h][d/h] learnable queries q_i, one per head */
  const void *w_o;         /* [d][d]   W^{o}                               */
  const void *b_o;         /* [d]                                          */
  const void *ln_o_gamma;  /* [d]                                          */
  const void *ln_o_beta;   /* [d]                                          */
  int32_t d_model;         /* d                                            */
  int32_t n_heads;         /* h (the paper uses 4)                         */
  float ln_eps;            /* LayerNorm epsilon (1e-5 when not trained otherwise) */
} umim_merge_weights;

/* A paged bf16 KV cache (layout in the header comment). */
typedef struct umim_paged_kv {
  void *base;         /* device pool                                   */
  int32_t n_layers;
  int32_t n_pages;    /* physical pages per layer                      */
  int32_t n_kv_heads;
  int32_t page_size;  /* must be UMIM_PAGE_SIZE                         */
  int32_t head_dim;   /* 64 or 128                                     */
} umim_paged_kv;

/* ------------------------------------------------------------------------
 * Merge module forward (Sec. 3.2 Eq. 1; App. C.1 full form):
 *   P   = LN_kv(GELU(E_s W_kv^T + b_kv)),  P = [P_1 .. P_h]
 *   a_i = softmax(P_i q_i / sqrt(d/h)),  o_i = a_i^T P_i
 *   z_s = LN_o(GELU(W_o [o_1; ..; o_h] + b_o))
 * GELU is the erf form, LayerNorm uses the biased variance.
 *
 * embeddings    device bf16 [vocab][d]  static embedding table e(.)
 * token_ids     device int32 [n_tokens] the span tokens, concatenated
 * span_offsets  device int32 [n_spans+1] CSR: span s = token_ids[off[s]..off[s+1])
 *               (1 <= off[s+1]-off[s] <= 4 is checked on the device)
 * surrogates    device fp32 [n_spans][d] output z_s
 * workspace     device, umim_merge_spans_workspace_size() bytes, 256-B aligned
 * Device-side errors: UMIM_ERR_INVALID_ARG for a token id outside [0, vocab)
 * (that token reads as zeros) or a malformed span (its z is then computed
 * from an all-zero pooled vector).
 * ------------------------------------------------------------------------ */
size_t umim_merge_spans_workspace_size(int64_t n_tokens, int32_t n_spans, int32_t d_model);

umim_status umim_merge_spans(const void *embeddings, int64_t vocab, const int32_t *token_ids,
                             int64_t n_tokens, const int32_t *span_offsets, int32_t n_spans,
                             const umim_merge_weights *weights, float *surrogates, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Compressed prompt (App. E "Prompt Merging", App. C.5, App. J.4): every
 * span of prompt b is replaced by bf16(z) (round to nearest even) and every
 * other token by its embedding row, in order; prompts are packed back to
 * back; position ids restart at 0 for every prompt (contiguous compressed
 * positions); cu_seqlens[b] is the first row of prompt b,
 * cu_seqlens[batch] = total rows = sum_b (L - sum (k - 1)).
 *
 * embeddings    device bf16 [vocab][d]
 * token_ids     device int32 [batch][prompt_len]
 * span_offsets  device int32 [batch+1] CSR over prompts
 * span_start    device int32 [n_spans] first position of each span inside its prompt
 * span_len      device int32 [n_spans] tokens per span (>= 1); spans of a prompt
 *               sorted, non-overlapping, inside the prompt
 * surrogates    device fp32 [n_spans][d] (as returned by umim_merge_spans)
 * out_embeds    device bf16 [out_capacity_rows][d]
 * position_ids  device int32 [out_capacity_rows]
 * cu_seqlens    device int32 [batch+1]
 * workspace     device, umim_build_compressed_workspace_size() bytes, 256-B
 *               aligned, zero-filled before its first use, then reused
 * Device-side errors: UMIM_ERR_INVALID_ARG for a bad span list or token id,
 * or when the compressed rows exceed out_capacity_rows (nothing is written
 * to out_embeds / position_ids then).
 * ------------------------------------------------------------------------ */
size_t umim_build_compressed_workspace_size(int32_t batch, int32_t n_spans);

umim_status umim_build_compressed(const void *embeddings, int64_t vocab, int32_t d_model,
                                  const int32_t *token_ids, int32_t batch, int32_t prompt_len,
                                  const int32_t *span_offsets, const int32_t *span_start,
                                  const int32_t *span_len, int32_t n_spans, const float *surrogates,
                                  void *out_embeds, int64_t out_capacity_rows, int32_t *position_ids,
                                  int32_t *cu_seqlens, void *workspace, size_t workspace_bytes,
                                  int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * KV-cache rollback and compaction (App. E "Decoding-Time Merging and
 * KV-Cache Update": the cached entries of a merged span are cropped and the
 * surrogate's single KV state takes their place, L' = L - (n-1) + 1; Fig. 2).
 * Generalised to any number of sorted, non-overlapping spans per sequence:
 * each span (s, k) of sequence b replaces its k stored entries, in every
 * layer, by one entry holding surrogate_k/v[span]; the entries after it
 * move left.  The result is written IN PLACE into the sequence's own pages
 * in logical order (new entry j -> page block_table[b][j/16], slot j%16).
 * Block-table entries p in [ceil(L'/16), ceil(L/16)) are reported in
 * freed_pages (sequence after sequence, ascending p) and set to -1;
 * seq_lens[b] becomes L' = L - sum (k - 1).  Slots at or after L' in the
 * last page keep unspecified contents.  Entries before a sequence's first
 * span are never read or written.
 *
 * kv            host struct describing the device pool (read and written)
 * block_table   device int32 [batch][max_pages], in/out
 * seq_lens      device int32 [batch], in/out
 * span_offsets  device int32 [batch+1] CSR over sequences
 * span_start    device int32 [n_spans] first replaced entry (logical index)
 * span_len      device int32 [n_spans] k = stored entries replaced (>= 1);
 *               the paper's n-1 when the newest token is not cached yet
 * surrogate_k/v device bf16 [n_spans][n_layers][n_kv_heads][head_dim]
 * freed_pages   device int32 [batch*max_pages] out, -1 terminated when not
 *               full; may be NULL
 * workspace     device, umim_kv_rollback_workspace_size() bytes, 256-B
 *               aligned, ZERO-FILLED BEFORE ITS FIRST USE and then reused
 *               unchanged between calls (it carries a call counter)
 * Preconditions checked on the device before anything is written (a
 * violation records UMIM_ERR_INVALID_ARG and leaves every buffer
 * untouched): 0 <= seq_lens[b] <= 16*max_pages; spans sorted,
 * non-overlapping, k >= 1, s >= 0, s + k <= seq_lens[b]; block-table
 * entries of used pages in [0, n_pages).  Not checked: that no physical
 * page is shared by two sequences.  UMIM_ERR_TIMEOUT leaves the cache
 * contents unspecified.
 * ------------------------------------------------------------------------ */
size_t umim_kv_rollback_workspace_size(int32_t batch, int32_t n_spans, int32_t max_pages, int32_t n_layers,
                                       int32_t n_kv_heads, int32_t head_dim);

umim_status umim_kv_rollback(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages,
                             int32_t *seq_lens, int32_t batch, const int32_t *span_offsets,
                             const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                             const void *surrogate_k, const void *surrogate_v, int32_t *freed_pages,
                             void *workspace, size_t workspace_bytes, int32_t *dev_status,
                             cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Position-aware rollback (App. J.4: a kept token at original position t
 * takes the compressed position pi(t) = t - r(t), r(t) the positions removed
 * before it; and its discussion of RoPE).  The cache holds keys already
 * rotated for their positions, so this variant of umim_kv_rollback also
 * rotates every moved kept entry's K rows (all layers and KV heads) by
 * -r(t) * rope_inv_freq[m] on the pairs (m, m + rotary_dim/2),
 * m < rotary_dim/2 (the half-split pairing of Llama-style RoPE):
 *   x' = x cos(r w_m) + y sin(r w_m),  y' = y cos(r w_m) - x sin(r w_m),
 * computed in fp32 and rounded to bf16 (nearest even), which gives each
 * moved key the rotation of its compressed position.  V rows, columns at or
 * beyond rotary_dim, surrogate entries (computed by the caller at their
 * compressed positions) and entries that do not move are unchanged; block
 * tables, lengths and freed pages are those of umim_kv_rollback.
 * rope_inv_freq  device fp32 [rotary_dim / 2]: the angular frequencies (any
 *                RoPE variant: base, scaling and all are folded into them)
 * rotary_dim     a multiple of 16, <= head_dim
 * Other arguments, workspace and errors: as umim_kv_rollback; a bad
 * rotary_dim or a NULL rope_inv_freq is UMIM_ERR_INVALID_ARG.
 * ------------------------------------------------------------------------ */
umim_status umim_kv_rollback_rope(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages,
                                  int32_t *seq_lens, int32_t batch, const int32_t *span_offsets,
                                  const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                                  const void *surrogate_k, const void *surrogate_v, const float *rope_inv_freq,
                                  int32_t rotary_dim, int32_t *freed_pages, void *workspace, size_t workspace_bytes,
                                  int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Decode-step KV append (App. E "Decoding-Time Merging and KV-Cache Update"
 * and Fig. 2 step (2): a generated token that completes no merge is
 * forwarded normally and one KV entry is appended).  For each sequence b
 * with L = seq_lens[b], in every layer, the K and V rows of entry L are
 * written to page block_table[b][L/16], slot L%16, from new_k/new_v[b];
 * when L % 16 == 0 that page is new_pages[b] (the caller's allocator picks
 * it) and is recorded in block_table[b][L/16]; seq_lens[b] becomes L + 1.
 * With merging, the decode loop appends first and then, when the suffix
 * matches a rule, rolls the last k stored entries back to one surrogate
 * entry with umim_kv_rollback (k counts the appended entry).
 *
 * kv            host struct describing the device pool (written)
 * block_table   device int32 [batch][max_pages], in/out
 * seq_lens      device int32 [batch], in/out
 * new_k/new_v   device bf16 [batch][n_layers][n_kv_heads][head_dim], 16-B aligned
 * new_pages     device int32 [batch] or NULL: read only for sequences whose
 *               length is a multiple of 16
 * dev_status    device int32 or NULL (device-side errors are then not
 *               reported)
 * No workspace.  Device-side errors: UMIM_ERR_INVALID_ARG, and that
 * sequence is left unchanged (the others are appended), when seq_lens[b] is
 * outside [0, 16*max_pages), or the destination page (new_pages[b] at a page
 * boundary, else block_table[b][L/16]) is outside [0, n_pages).  Not
 * checked: that the new page is free.
 * ------------------------------------------------------------------------ */
umim_status umim_kv_append(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                           int32_t batch, const void *new_k, const void *new_v, const int32_t *new_pages,
                           int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Decode step with decoding-time merging (App. E "Decoding-Time Merging and
 * KV-Cache Update"; Fig. 2 steps (2) and (3)): after each generated token
 * the recent suffix is checked against the merge rules; without a match the
 * token's KV entry is appended, with a match the n-gram's cached entries are
 * cropped and the surrogate's single KV entry takes their place.  One call
 * does both for a batch, in place, per sequence b with L = seq_lens[b]:
 *   merge_k[b] == 0 (or merge_k NULL): new_k/new_v[b] are appended at slot L
 *     exactly as umim_kv_append does (new_pages[b] opens the page when
 *     L % 16 == 0);
 *   merge_k[b] = k in [1, 16]: the new token and the k - 1 stored entries
 *     before it form the merged span, so surrogate row merge_row[b] is
 *     written at slot s = L + 1 - k in every layer, seq_lens[b] becomes
 *     s + 1, and the one page that no longer holds an entry, if any (the
 *     page the append would have opened included), is set to -1 in the block
 *     table and reported in released_pages[b] (-1 otherwise).
 * The result is identical to umim_kv_append followed by umim_kv_rollback of
 * the suffix spans (s, k); no entry moves, since a suffix has nothing after
 * it.  k counts stored entries after the append, i.e. the paper's n.
 *
 * new_k/new_v       device bf16 [batch][n_layers][n_kv_heads][head_dim]
 * new_pages         device int32 [batch] or NULL (read at page boundaries)
 * merge_k           device int32 [batch] or NULL (no merges)
 * merge_row         device int32 [batch]: row of the surrogate arrays for a
 *                   merging sequence
 * surrogate_k/v     device bf16 [n_merge_rows][n_layers][n_kv_heads][head_dim]
 * released_pages    device int32 [batch] out, or NULL
 * No workspace.  Device-side errors: UMIM_ERR_INVALID_ARG, and that sequence
 * is left unchanged, when seq_lens[b] is outside [0, 16*max_pages), k is
 * outside [0, min(16, L + 1)], merge_row[b] is outside [0, n_merge_rows), or
 * a page to write is outside [0, n_pages).
 * ------------------------------------------------------------------------ */
umim_status umim_decode_append_merge(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages,
                                     int32_t *seq_lens, int32_t batch, const void *new_k, const void *new_v,
                                     const int32_t *new_pages, const int32_t *merge_k, const int32_t *merge_row,
                                     int32_t n_merge_rows, const void *surrogate_k, const void *surrogate_v,
                                     int32_t *released_pages, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * One layer of a decode step with decoding-time merging, in one launch
 * (App. E "Decoding-Time Merging and KV-Cache Update"; Fig. 2 steps (2) and
 * (3); App. I.1 on the overhead of many small kernel launches per step).
 * A forward pass produces layer l's new K/V entry only after layer l - 1's
 * attention, so a decode step calls this once per layer, in layer order,
 * with that layer's new entries, query and (for merging sequences)
 * surrogate entries.  Per sequence b, with L = seq_lens[b] as it was before
 * the step and k = merge_k[b] (0 when merge_k is NULL):
 *   k == 0      the new entry new_k/new_v[b] is written at slot s = L
 *               (at a page boundary into page new_pages[b]);
 *   k in 1..16  the forwarded token completes a merge of the last k tokens
 *               (the k - 1 cached entries before it and itself): surrogate
 *               row merge_row[b] is written at slot s = L + 1 - k;
 * and out[b] is decode attention of q[b] over slots [0, s] of layer `layer`
 * (the entry just written included).  Layer by layer this equals
 * umim_decode_append_merge followed by umim_decode_attention.
 * Block tables and lengths are read, not changed, by every call of the step
 * except the one with `commit` != 0, which must be the step's last call (its
 * last layer): once every CTA of that launch has finished reading them, it
 * records new_pages[b] in the block table when L % 16 == 0, releases the
 * page that no longer holds an entry (set to -1, reported in
 * released_pages[b], -1 if none; at most one) and sets seq_lens[b] = s + 1.
 *
 * q                 device bf16 [batch][n_q_heads][head_dim] (this layer)
 * new_k/new_v       device bf16: row b at new_k + b * new_row_stride elements,
 *                   n_kv_heads * head_dim values (this layer), 16-B aligned;
 *                   new_row_stride 0 means n_kv_heads * head_dim, otherwise a
 *                   multiple of 8 not below it (rows inside a fused QKV
 *                   projection output, or one layer of a [batch][layers][...]
 *                   array)
 * new_pages         device int32 [batch] or NULL (read at page boundaries)
 * merge_k, merge_row  device int32 [batch] or NULL (no merges)
 * surrogate_k/v     device bf16 [n_merge_rows][n_kv_heads][head_dim] (this layer)
 * released_pages    device int32 [batch] out (commit call), or NULL
 * out               device bf16 [batch][n_q_heads][head_dim], 4-B aligned
 * workspace         device, umim_decode_layer_step_workspace_size() bytes,
 *                   256-B aligned, ZEROED before its first use; each call
 *                   leaves it ready for the next.  After a call that reported
 *                   UMIM_ERR_TIMEOUT, zero it again.  Calls sharing one
 *                   workspace must not overlap on the GPU.
 * Host-side errors: UMIM_ERR_UNSUPPORTED for batch > 4096 or the shapes
 * umim_decode_attention does not support.  Device-side errors:
 * UMIM_ERR_INVALID_ARG when seq_lens[b] is outside [0, 16*max_pages), k is
 * outside [0, min(16, L + 1)], merge_row[b] is outside [0, n_merge_rows), or
 * a page to write is outside [0, n_pages): that sequence is left unchanged
 * (nothing written, not committed) and its output is attention over its
 * unchanged cache; UMIM_ERR_TIMEOUT for a stalled copy.
 * ------------------------------------------------------------------------ */
size_t umim_decode_layer_step_workspace_size(int32_t batch, int32_t n_kv_heads, int32_t head_dim);

umim_status umim_decode_layer_step(const void *q, int32_t n_q_heads, const umim_paged_kv *kv, int32_t layer,
                                   int32_t *block_table, int32_t max_pages, int32_t *seq_lens, int32_t batch,
                                   const void *new_k, const void *new_v, int64_t new_row_stride,
                                   const int32_t *new_pages, const int32_t *merge_k, const int32_t *merge_row,
                                   int32_t n_merge_rows, const void *surrogate_k, const void *surrogate_v,
                                   int32_t commit, int32_t *released_pages, float scale, void *out, void *workspace,
                                   size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Grouped-query decode attention over the (compacted) paged cache, one
 * query token per sequence (App. I.1; the backbone's ordinary attention):
 *   out[b][h] = sum_{j < seq_lens[b]} softmax_j(scale <q[b][h], K[b][g][j]>) V[b][g][j]
 *   g = h / (n_q_heads / n_kv_heads),  scale = 1/sqrt(head_dim) when 0 is given.
 * A sequence with seq_lens[b] == 0 gets a zero output.  Reads only: the
 * cache, block table and lengths are not modified.
 *
 * q             device bf16 [batch][n_q_heads][head_dim]
 * kv, layer     cache and the layer to read
 * block_table   device int32 [batch][max_pages]
 * seq_lens      device int32 [batch]
 * out           device bf16 [batch][n_q_heads][head_dim]
 * workspace     device, umim_decode_attention_workspace_size() bytes, 256-B aligned
 * Device-side errors: UMIM_ERR_INVALID_ARG for seq_lens[b] outside
 * [0, 16*max_pages] or a used block-table entry outside [0, n_pages)
 * (that page reads as zeros), UMIM_ERR_TIMEOUT for a stalled copy.
 * ------------------------------------------------------------------------ */
size_t umim_decode_attention_workspace_size(int32_t batch, int32_t n_q_heads, int32_t n_kv_heads,
                                            int32_t head_dim);

umim_status umim_decode_attention(const void *q, int32_t n_q_heads, const umim_paged_kv *kv, int32_t layer,
                                  const int32_t *block_table, int32_t max_pages, const int32_t *seq_lens,
                                  int32_t batch, float scale, void *out, void *workspace,
                                  size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Prefill attention over packed compressed prompts (App. E "Prompt
 * Merging", App. C.5: the compressed embeddings, with contiguous positions,
 * go through the frozen backbone's prefill, whose causal self-attention then
 * runs over the shorter sequences).  Sequence b owns rows cu_seqlens[b] ..
 * cu_seqlens[b+1]-1 (the cu_seqlens umim_build_compressed writes); per
 * sequence, with rows i, j counted inside it:
 *   out[i, h] = sum_{j <= i} softmax_j(scale <q[i, h], k[j, g]>) v[j, g],
 *   g = h / (n_q_heads / n_kv_heads),  scale = 1/sqrt(head_dim) if scale <= 0.
 * Rotary embeddings are already applied to q and k by the caller.
 * q            device bf16 [n_rows][n_q_heads][head_dim], 16-B aligned
 * k, v         device bf16 [n_rows][n_kv_heads][head_dim], 16-B aligned
 * cu_seqlens   device int32 [batch + 1], cu_seqlens[0] = 0, nondecreasing,
 *              cu_seqlens[batch] <= n_rows
 * out          device bf16 [n_rows][n_q_heads][head_dim] (rows outside every
 *              sequence are not written)
 * workspace    device, umim_prefill_attention_workspace_size() bytes, 256-B
 *              aligned (it holds the tile plan and a transposed copy of v,
 *              each sequence padded to 64 keys: about
 *              n_kv_heads * head_dim * (n_rows + 64 * batch) * 2 bytes)
 * head_dim 64 or 128; n_q_heads a multiple of n_kv_heads (else
 * UMIM_ERR_UNSUPPORTED).  Device-side errors: UMIM_ERR_INVALID_ARG for
 * offsets that break the rules above (nothing is written);
 * UMIM_ERR_UNSUPPORTED when some |v| >= 65504 or is not finite (the P V
 * product runs on fp16 operands; the output is then not valid).
 * ------------------------------------------------------------------------ */
size_t umim_prefill_attention_workspace_size(int32_t batch, int32_t n_rows, int32_t n_kv_heads, int32_t head_dim);

umim_status umim_prefill_attention(const void *q, const void *k, const void *v, int32_t n_rows, int32_t n_q_heads,
                                   int32_t n_kv_heads, int32_t head_dim, const int32_t *cu_seqlens, int32_t batch,
                                   float scale, void *out, void *workspace, size_t workspace_bytes,
                                   int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Merge rules (App. E "Rule Matching").  A rule is a token n-gram, n in
 * {2, 3, 4}; its rule id is its row in the list given to umim_rules_build.
 * The table is open addressing over 16-byte slots (the n-gram packed as four
 * 24-bit token ids, and the rule id) in a caller-owned device buffer.
 *
 * umim_rule_table_bytes: buffer size for n_rules rules (a power of two times
 * 16 bytes, at least 24 * n_rules: load factor <= 2/3; 64 MB for the 2.2
 * million rules of a Llama-3 rule set, which then stays in L2).
 *
 * umim_rules_build: fills the table.
 * table         device, table_bytes (16 times a power of two, >= 24 *
 *               n_rules and >= 256), 16-B aligned; overwritten
 * rule_tokens   device int32 [n_rules][4], 16-B aligned: the n token ids of
 *               a rule (each in [0, 0xFFFFFF)) followed by 4 - n entries -1
 * Device-side errors: UMIM_ERR_INVALID_ARG when a rule row is malformed or
 * an n-gram occurs twice (the table is then not usable).  Token ids are
 * limited to 24 bits (every published vocabulary fits).
 * ------------------------------------------------------------------------ */
size_t umim_rule_table_bytes(int64_t n_rules);

umim_status umim_rules_build(void *table, size_t table_bytes, const int32_t *rule_tokens, int64_t n_rules,
                             int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Prompt merging's span selection (App. E "Rule Matching", "Prompt
 * Merging"): each prompt is scanned from left to right; at a position the
 * 4-, 3- and then 2-gram starting there is tested and the first that is a
 * rule becomes a span, the scan continuing after it; otherwise the scan moves
 * on by one token.  Output: the spans as the CSR that umim_build_compressed
 * takes, each span's rule id (the row of a surrogate lookup table), and
 * optionally the span tokens as the CSR that umim_merge_spans takes.
 *
 * token_ids       device int32 [batch][max_len]; tokens past a prompt's
 *                 length are not read
 * prompt_lens     device int32 [batch], each in [0, max_len], or NULL (all
 *                 max_len)
 * span_offsets    device int32 [batch + 1] out: spans of prompt b are
 *                 span_offsets[b] .. span_offsets[b+1]-1
 * span_start      device int32 [batch * (max_len/2)] out: start, relative to
 *                 the prompt (capacity: a prompt of length L has at most L/2)
 * span_len        device int32, same capacity: n
 * span_rule       device int32, same capacity: rule id
 * merge_token_ids device int32 [batch * max_len] out, or NULL: the tokens of
 *                 every span, span after span
 * merge_offsets   device int32 [batch * (max_len/2) + 1] out (with
 *                 merge_token_ids): CSR offsets of the spans' tokens
 * workspace       device, umim_match_prompts_workspace_size() bytes, 256-B
 *                 aligned
 * Host-side errors: batch * max_len >= 2^31.  Device-side errors:
 * UMIM_ERR_INVALID_ARG for a prompt length outside [0, max_len] (clamped) or
 * a token id outside [0, 0xFFFFFF) (no n-gram containing it matches).
 * ------------------------------------------------------------------------ */
size_t umim_match_prompts_workspace_size(int32_t batch, int32_t max_len);

umim_status umim_match_prompts(const void *table, size_t table_bytes, const int32_t *token_ids, int32_t batch,
                               int32_t max_len, const int32_t *prompt_lens, int32_t *span_offsets,
                               int32_t *span_start, int32_t *span_len, int32_t *span_rule,
                               int32_t *merge_token_ids, int32_t *merge_offsets, void *workspace,
                               size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Decoding-time span selection (App. E "Rule Matching", "Decoding-Time
 * Merging"): after each generated token, the raw-token suffix ending at it is
 * tested longest first (4, 3, 2 tokens).  A merged span counts as one marker
 * that no later suffix includes, and generation starts with an empty suffix
 * (the prompt is not part of it).  Per sequence the state is the last up to
 * three raw generated tokens:
 *   typedef: int32 raw[3] (right-aligned: the last n_raw entries are the
 *   suffix, oldest first), int32 n_raw in [0, 3].  A zeroed state is the
 *   start of generation.
 * Per sequence b, for new_tokens[b]:
 *   merge_k[b]    n of the merge it completes (the k of
 *                 umim_decode_append_merge), or 0
 *   merge_rule[b] its rule id, or -1
 *   merge_row[b]  its rank among this step's merging sequences (in sequence
 *                 order), or -1: the row of the surrogate arrays that
 *                 umim_decode_append_merge reads
 *   rows_rule     device int32 [batch] out, or NULL: rule id of each row
 *   n_merges      device int32 [1] out, or NULL: number of merging sequences
 * state is updated in place.  Device-side errors: UMIM_ERR_INVALID_ARG for
 * n_raw outside [0, 3] (read as 0) or a token outside [0, 0xFFFFFF) (no
 * merge; the suffix restarts after it).
 * ------------------------------------------------------------------------ */
typedef struct {
  int32_t raw[3];
  int32_t n_raw;
} umim_suffix_state;

umim_status umim_match_suffix(const void *table, size_t table_bytes, umim_suffix_state *state,
                              const int32_t *new_tokens, int32_t batch, int32_t *merge_k, int32_t *merge_rule,
                              int32_t *merge_row, int32_t *rows_rule, int32_t *n_merges, int32_t *dev_status,
                              cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Surrogate lookup (App. E, potential engineering optimizations): a
 * surrogate depends only on its span's tokens, so one per rule can be
 * computed ahead of time (umim_merge_spans over the rules' n-grams) and
 * fetched by rule id instead of running the merge module.
 * lut        device fp32 [n_rules][d], 16-B aligned (d a multiple of 4)
 * rule_ids   device int32 [n_max]
 * n_dev      device int32 [1] or NULL: rows to fetch, min(*n_dev, n_max)
 *            (e.g. span_offsets[batch] of umim_match_prompts); NULL: n_max
 * out        device fp32 [n_max][d], 16-B aligned
 * Device-side errors: UMIM_ERR_INVALID_ARG for a rule id outside
 * [0, n_rules) (that row is written as zeros).
 * ------------------------------------------------------------------------ */
umim_status umim_lookup_surrogates(const float *lut, int64_t n_rules, int32_t d, const int32_t *rule_ids,
                                   int32_t n_max, const int32_t *n_dev, float *out, int32_t *dev_status,
                                   cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Aligned predictive distillation, the training objective of the merge
 * module (App. F "Predictive Distillation Loss and Alignment Metrics",
 * Algorithm 1 and the masked distillation loss).  The frozen backbone runs on
 * the original sequences (teacher) and on the compressed ones (student); the
 * two calls below pair their rows and compute the loss and its gradient with
 * respect to the student logits.
 *
 * umim_distill_align: the masks and Pack of Algorithm 1 as row indices.  For
 * sample b with original length L_b and sorted, non-overlapping spans
 * (s_i, n_i), the keep mask marks every retained token and, for each span,
 * only its last position s_i + n_i - 1; the teacher mask is the keep mask
 * from the first span's start s_b on (N_b = its number of ones); the student
 * mask marks the last N_b positions of the compressed sequence (length
 * L~_b = L_b - sum (n_i - 1)); Pack pairs them in order.  A sample without
 * spans has no pairs.  Rows are numbered over the packed batches: teacher
 * row of (b, t) = sum_{b'<b} L_b' + t; student row of (b, j) =
 * sum_{b'<b} L~_b' + j, the row order of umim_build_compressed's output.
 * seq_lens      device int32 [batch] L_b
 * span_offsets  device int32 [batch + 1] CSR over the spans; span_start /
 *               span_len device int32 [n_spans], start relative to the sample
 * pair_offsets  device int32 [batch + 1] out: pairs of sample b are
 *               pair_offsets[b] .. pair_offsets[b+1]-1, in Pack order
 * teacher_rows, student_rows  device int32 [capacity] out
 * student_cu    device int32 [batch + 1] out, or NULL: prefix sums of L~_b
 * workspace     device, umim_distill_align_workspace_size() bytes, 256-B
 *               aligned, zero-filled before its first use
 * Device-side errors: UMIM_ERR_INVALID_ARG (nothing written) for spans that
 * are unsorted, overlap, are empty or pass L_b, a negative length, bad
 * offsets, more pairs than capacity or more than 2^31 - 1 teacher rows.
 *
 * umim_distill_soft_ce: over the N aligned pairs (teacher row t_k, student
 * row s_k), with P = softmax over the whole vocabulary of a logits row,
 *   loss = -(1/N) sum_k sum_v P^T_k(v) log(P^S_k(v) + eps)
 * and the gradient with respect to the student logits of row s_k
 *   -(1/N) (a_v - P^S_k(v) sum_u a_u),  a_u = P^T_k(u) P^S_k(u) / (P^S_k(u) + eps);
 * student rows in no pair have a zero gradient.  Computed in fp32 from bf16
 * logits; each logit is read once.
 * teacher_logits  device bf16 [n_teacher_rows][ld], 16-B aligned
 * student_logits  device bf16 [n_student_rows][ld], 16-B aligned
 * vocab, ld       vocabulary size (1 .. 163840) and row stride in elements
 *                 (a multiple of 8, >= vocab rounded up to a multiple of 8;
 *                 the elements from vocab up to that are read, never used)
 * teacher_rows, student_rows  device int32 [max_pairs] (e.g. from
 *                 umim_distill_align); each student row at most once
 * n_pairs         device int32 [1] or NULL: N (NULL: N = max_pairs), e.g.
 *                 pair_offsets + batch of umim_distill_align
 * eps             the loss's stability constant (>= 0, finite)
 * loss            device fp32 [1] out
 * pair_loss       device fp32 [max_pairs] out, or NULL: each pair's
 *                 -sum_v P^T log(P^S + eps)
 * grad            device bf16 [n_student_rows][ld] out, or NULL (loss only);
 *                 elements [0, vocab) of every row written
 * workspace       device, umim_distill_soft_ce_workspace_size() bytes, 256-B
 *                 aligned (no initial contents required)
 * Host-side errors: UMIM_ERR_UNSUPPORTED for a vocabulary above 163840.
 * Device-side errors: UMIM_ERR_INVALID_ARG (nothing written) for N outside
 * [0, max_pairs], a row outside its logits or a student row in two pairs.
 * ------------------------------------------------------------------------ */
size_t umim_distill_align_workspace_size(int32_t batch, int32_t n_spans);

umim_status umim_distill_align(const int32_t *seq_lens, int32_t batch, const int32_t *span_offsets,
                               const int32_t *span_start, const int32_t *span_len, int32_t n_spans,
                               int32_t *pair_offsets, int32_t *teacher_rows, int32_t *student_rows,
                               int32_t capacity, int32_t *student_cu, void *workspace, size_t workspace_bytes,
                               int32_t *dev_status, cudaStream_t stream);

size_t umim_distill_soft_ce_workspace_size(int32_t n_student_rows, int32_t max_pairs);

umim_status umim_distill_soft_ce(const void *teacher_logits, int32_t n_teacher_rows, const void *student_logits,
                                 int32_t n_student_rows, int32_t vocab, int64_t ld, const int32_t *teacher_rows,
                                 const int32_t *student_rows, int32_t max_pairs, const int32_t *n_pairs, float eps,
                                 float *loss, float *pair_loss, void *grad, void *workspace,
                                 size_t workspace_bytes, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Decode attention for callers that cannot allocate GPU memory.
 * The paper has no counterpart to this call; it is a convenience of this
 * library.  A serving engine that gives all device memory to its own block
 * allocator up front, or a plug-in running inside another framework that
 * forbids allocations outside its arena, may be unable to provide the
 * workspace that umim_decode_attention needs.  This variant computes exactly
 * the same result but takes its scratch (split-K plan and fp32 partials)
 * from an array of UMIM_STATIC_SCRATCH_BYTES compiled into the library.
 *  - Arguments and results are those of umim_decode_attention, without the
 *    workspace.  It calls no cudaMalloc, cudaFree or allocating library
 *    routine.
 *  - A batch whose scratch would exceed the array (about
 *    (batch * n_kv_heads + 12 * SMs) * 16 * (head_dim + 2) * 4 bytes) is
 *    rejected with UMIM_ERR_WORKSPACE before anything is launched.
 *  - The first call on a device does the set-up: it looks up the array's
 *    device address (cudaGetSymbolAddress) and the SM count.  Under CUDA's
 *    default lazy module loading, that lookup is also when the driver loads
 *    the array onto the device and reserves its UMIM_STATIC_SCRATCH_BYTES,
 *    which then stay reserved until the process exits.  So make the first
 *    call on each device early: before the caller's own allocator takes the
 *    device's free memory (otherwise the set-up fails with UMIM_ERR_CUDA),
 *    and before any stream capture begins.  Later calls reserve nothing.
 *  - The stream's device is made current for the call and the caller's
 *    current device is restored before it returns.  While the stream is
 *    being captured into a CUDA graph its device cannot be queried, so the
 *    current device must then be the stream's device.
 *  - All calls share the one array.  Nothing in it has to start at zero
 *    (each call rewrites every field it reads), but calls whose kernels
 *    overlap on the GPU (different streams, no ordering between them) race
 *    on it and give wrong results: order such calls on one stream.
 * ------------------------------------------------------------------------ */
#define UMIM_STATIC_SCRATCH_BYTES (32u << 20)

umim_status umim_decode_attention_static(const void *q, int32_t n_q_heads, const umim_paged_kv *kv,
                                         int32_t layer, const int32_t *block_table, int32_t max_pages,
                                         const int32_t *seq_lens, int32_t batch, float scale, void *out,
                                         int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Self-test of the bounded waits (not part of the method).  Every wait of
 * the library on another agent (an mbarrier completed by TMA or the tensor
 * cores, a counter raised by another CTA) gives up after a time limit (1 s
 * inside the calls above), records UMIM_ERR_TIMEOUT in the status word and
 * returns, so the context stays usable.  This call waits, with limit_us
 * (1 .. 1e6) microseconds, on something that never happens:
 *   which 0: an mbarrier that nobody arrives on;
 *   which 1: flags[0] >= 1 with flags[1] as the abort word (the rollback
 *            movers' wait); the caller keeps both at 0.
 * flags       device int32 [2] (which 1) or NULL
 * elapsed_ns  device uint64 [1] out, or NULL: how long the wait lasted
 * The expected outcome is UMIM_ERR_TIMEOUT in dev_status.
 * ------------------------------------------------------------------------ */
umim_status umim_selftest_bounded_wait(int32_t which, uint32_t limit_us, const int32_t *flags,
                                       uint64_t *elapsed_ns, int32_t *dev_status, cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Debug build (not part of the method).  libumim_debug.so is this library
 * compiled with UMIM_DEBUG defined: every kernel also checks, where it loads
 * or stores, that each index it computed from device data (a page from a
 * block table, a row or offset from one of its own plans, a partial-result
 * slot) lies inside the buffer it addresses.  A failed check records
 * UMIM_ERR_BOUNDS | site << 8 in dev_status (first error wins), skips that
 * access (a store is dropped, a load reads zeros) and the kernel carries
 * on; the call's outputs are then unspecified.  These are checks of the
 * library's own invariants: inputs are validated the same way in both
 * builds, so on valid and invalid inputs alike a correct library never
 * records UMIM_ERR_BOUNDS.  The calls and their results are otherwise
 * identical to libumim.so's.
 *
 * umim_debug_build       1 in libumim_debug.so, 0 in libumim.so
 * umim_debug_site_name   the name of the access site in bits 8.. of a status
 *                        word ("" when there is none)
 * umim_selftest_bounds_check
 *                        one check of the mechanism: a kernel stores 1 into
 *                        buf[index] if 0 <= index < n, through the same
 *                        check as the other kernels' access sites.  buf is
 *                        a device int32 [n].  With an index outside [0, n)
 *                        the expected outcome is UMIM_ERR_BOUNDS | 1 << 8 in
 *                        dev_status and buf unchanged.  In libumim.so it
 *                        returns UMIM_ERR_UNSUPPORTED and launches nothing.
 * ------------------------------------------------------------------------ */
int umim_debug_build(void);
const char *umim_debug_site_name(int32_t status);
umim_status umim_selftest_bounds_check(int32_t *buf, int64_t n, int64_t index, int32_t *dev_status,
                                       cudaStream_t stream);

/* ------------------------------------------------------------------------
 * Kernel tracing, for profiling (not part of the method).  Between
 * umim_trace_start and umim_trace_stop every call above records a CUDA
 * event on its stream before each kernel it launches and one after its last
 * kernel, so consecutive events bracket one kernel.  The library creates the
 * events itself (no device memory).  Process-wide and not thread-safe.
 *
 * umim_trace_start  begin recording, at most `capacity` events; returns
 *                   UMIM_ERR_CUDA if the events cannot be created
 * umim_trace_stop   stop recording (the recorded events are kept)
 * umim_trace_read   synchronise on the last event, write up to `cap` kernel
 *                   durations (ms) and their labels (static strings) in
 *                   launch order; returns how many were written
 * ------------------------------------------------------------------------ */
umim_status umim_trace_start(int32_t capacity);
void umim_trace_stop(void);
int32_t umim_trace_read(float *ms, const char **labels, int32_t cap);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* UMIM_H_ */
