"""Python binding of libumim (GB300 / sm_103a), the decode step over a merged
context of UMIM (arXiv 2609.27233).

Thin argument marshalling only: every step runs in the library's CUDA
kernels.  PyTorch provides device memory and the current stream.  The entry
points keep the C names:

  umim_merge_spans        merge module M_phi (Sec. 3.2 Eq. 1, App. C.1)
  umim_build_compressed   compressed prompt embeddings + positions (App. E, App. C.5)
  umim_kv_rollback        KV-cache rollback and in-place compaction (App. E, Fig. 2)
  umim_kv_append          decode-step append of one KV entry per layer (App. E, Fig. 2)
  umim_decode_append_merge  append or suffix merge per sequence in one call (App. E decoding loop)
  umim_decode_attention   GQA decode attention over the compacted paged cache (App. I.1)
  umim_decode_layer_step  one layer of a decode step: its new or surrogate entry written and
                          attention over the updated cache in one launch (App. E, App. I.1)
  umim_prefill_attention  causal GQA attention over the packed compressed prompts (App. E, App. C.5)
  umim_rules_build, umim_match_prompts, umim_match_suffix, umim_lookup_surrogates
                          merge-rule table, longest-first span selection for prompts
                          and for decoding, and precomputed surrogates by rule id (App. E)
  umim_distill_align, umim_distill_soft_ce
                          aligned predictive distillation: teacher/student row pairing
                          and the full-vocabulary soft-target cross-entropy with its
                          gradient (App. F, Algorithm 1)
"""
import ctypes

import torch

from . import _lib
from ._lib import MergeWeightsC, PagedKVC

UMIM_OK = 0
STATUS = {0: "UMIM_OK", 1: "UMIM_ERR_INVALID_ARG", 2: "UMIM_ERR_UNSUPPORTED", 3: "UMIM_ERR_CUDA",
          4: "UMIM_ERR_TIMEOUT", 5: "UMIM_ERR_WORKSPACE", 6: "UMIM_ERR_BOUNDS"}
UMIM_ERR_BOUNDS = 6   # debug build: the status word holds 6 | site << 8
PAGE_SIZE = 16
STATIC_SCRATCH_BYTES = 32 << 20   # UMIM_STATIC_SCRATCH_BYTES of include/umim.h


class UmimError(RuntimeError):
    def __init__(self, code, where=""):
        self.code = int(code)
        self.site = ""
        msg = STATUS.get(self.code, self.code)
        if self.code & 0xff == UMIM_ERR_BOUNDS:   # the debug build's access-site checks
            self.site = lib().umim_debug_site_name(self.code).decode()
            msg = f"UMIM_ERR_BOUNDS at {self.site}"
        super().__init__(f"{where}: {msg}")


def use_debug_library(flag: bool = True) -> None:
    """Run every later call on libumim_debug.so, the build whose kernels check
    each index they compute at their access sites (or back on libumim.so)."""
    _lib.use_debug(flag)


def lib():
    return _lib.load()


def _p(t):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code, where):
    if code != UMIM_OK:
        raise UmimError(code, where)


def _dev(t):
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    return t.device


def new_status(device):
    """A zeroed device int32 that receives device-side errors."""
    return torch.zeros(1, dtype=torch.int32, device=device)


def check_status(dev_status, where="device"):
    v = int(dev_status.item())
    if v != UMIM_OK:
        raise UmimError(v, where)


def workspace(nbytes, device):
    """A zero-filled, 256-byte aligned device workspace of at least nbytes."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def paged_kv(pool):
    """umim_paged_kv for a bf16 pool shaped [layers][pages][2][Hkv][16][D]."""
    if pool.dtype != torch.bfloat16 or pool.dim() != 6 or pool.shape[2] != 2 or not pool.is_contiguous():
        raise ValueError("pool must be contiguous bf16 [layers][pages][2][Hkv][16][D]")
    return PagedKVC(pool.data_ptr(), pool.shape[0], pool.shape[1], pool.shape[3], pool.shape[4], pool.shape[5])


def merge_weights_c(w):
    g = (lambda k: getattr(w, k)) if not isinstance(w, dict) else (lambda k: w[k])
    names = ("w_kv", "b_kv", "ln_kv_gamma", "ln_kv_beta", "query", "w_o", "b_o", "ln_o_gamma", "ln_o_beta")
    for k in names:
        t = g(k)
        if t.dtype != torch.bfloat16 or not t.is_contiguous():
            raise ValueError(f"merge weight {k} must be contiguous bf16")
    return MergeWeightsC(*[g(k).data_ptr() for k in names], int(g("d_model")), int(g("n_heads")),
                         float(g("ln_eps")))


# ---------------------------------------------------------------------------
# workspace sizes
# ---------------------------------------------------------------------------
def umim_merge_spans_workspace_size(n_tokens, n_spans, d_model):
    return int(lib().umim_merge_spans_workspace_size(n_tokens, n_spans, d_model))


def umim_build_compressed_workspace_size(batch, n_spans):
    return int(lib().umim_build_compressed_workspace_size(batch, n_spans))


def umim_kv_rollback_workspace_size(batch, n_spans, max_pages, n_layers, n_kv_heads, head_dim):
    return int(lib().umim_kv_rollback_workspace_size(batch, n_spans, max_pages, n_layers, n_kv_heads, head_dim))


def umim_prefill_attention_workspace_size(batch, n_rows, n_kv_heads, head_dim):
    return int(lib().umim_prefill_attention_workspace_size(batch, n_rows, n_kv_heads, head_dim))


def umim_decode_attention_workspace_size(batch, n_q_heads, n_kv_heads, head_dim):
    return int(lib().umim_decode_attention_workspace_size(batch, n_q_heads, n_kv_heads, head_dim))


# ---------------------------------------------------------------------------
# the calls
# ---------------------------------------------------------------------------
def umim_merge_spans(embeddings, token_ids, span_offsets, weights, surrogates=None, workspace_buf=None,
                     dev_status=None, stream=None):
    """Surrogate embeddings z (fp32 [S][d]) of the spans in CSR form."""
    dev = _dev(embeddings)
    d = embeddings.shape[1]
    S = span_offsets.numel() - 1
    T = token_ids.numel()
    if surrogates is None:
        surrogates = torch.empty((S, d), dtype=torch.float32, device=dev)
    if workspace_buf is None:
        workspace_buf = workspace(umim_merge_spans_workspace_size(T, S, d), dev)
    wc = merge_weights_c(weights)
    code = lib().umim_merge_spans(_p(embeddings), embeddings.shape[0], _p(token_ids), T, _p(span_offsets), S,
                                  ctypes.byref(wc), _p(surrogates), _p(workspace_buf), workspace_buf.numel(),
                                  _p(dev_status), _stream(stream))
    _check(code, "umim_merge_spans")
    return surrogates


def umim_build_compressed(embeddings, token_ids, span_offsets, span_start, span_len, surrogates,
                          out_embeds=None, position_ids=None, cu_seqlens=None, workspace_buf=None,
                          dev_status=None, stream=None):
    """(out_embeds [rows][d] bf16, position_ids [rows], cu_seqlens [B+1]); the
    first cu_seqlens[-1] rows are the packed compressed prompts."""
    dev = _dev(embeddings)
    B, L = token_ids.shape
    d = embeddings.shape[1]
    S = span_start.numel()
    if out_embeds is None:
        out_embeds = torch.empty((B * L, d), dtype=torch.bfloat16, device=dev)
    if position_ids is None:
        position_ids = torch.empty(out_embeds.shape[0], dtype=torch.int32, device=dev)
    if cu_seqlens is None:
        cu_seqlens = torch.empty(B + 1, dtype=torch.int32, device=dev)
    if workspace_buf is None:
        workspace_buf = workspace(umim_build_compressed_workspace_size(B, S), dev)
    code = lib().umim_build_compressed(_p(embeddings), embeddings.shape[0], d, _p(token_ids), B, L,
                                       _p(span_offsets), _p(span_start), _p(span_len), S, _p(surrogates),
                                       _p(out_embeds), out_embeds.shape[0], _p(position_ids), _p(cu_seqlens),
                                       _p(workspace_buf), workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_build_compressed")
    return out_embeds, position_ids, cu_seqlens


def umim_kv_rollback(pool, block_table, seq_lens, span_offsets, span_start, span_len, surrogate_k, surrogate_v,
                     freed_pages=None, workspace_buf=None, dev_status=None, stream=None, rope_inv_freq=None,
                     rotary_dim=None):
    """In-place rollback of pool / block_table / seq_lens; returns freed_pages
    (device int32 [B*max_pages], -1 terminated).  With rope_inv_freq (device
    fp32 [rotary_dim/2]) moved keys are re-rotated to their compressed
    positions (umim_kv_rollback_rope)."""
    dev = _dev(pool)
    kv = paged_kv(pool)
    B, max_pages = block_table.shape
    S = span_start.numel()
    if freed_pages is None:
        freed_pages = torch.empty(max(1, B * max_pages), dtype=torch.int32, device=dev)
    if workspace_buf is None:
        workspace_buf = workspace(umim_kv_rollback_workspace_size(B, S, max_pages, kv.n_layers, kv.n_kv_heads,
                                                                  kv.head_dim), dev)
    if rope_inv_freq is None:
        code = lib().umim_kv_rollback(ctypes.byref(kv), _p(block_table), max_pages, _p(seq_lens), B,
                                      _p(span_offsets), _p(span_start), _p(span_len), S, _p(surrogate_k),
                                      _p(surrogate_v), _p(freed_pages), _p(workspace_buf), workspace_buf.numel(),
                                      _p(dev_status), _stream(stream))
        _check(code, "umim_kv_rollback")
    else:
        rd = kv.head_dim if rotary_dim is None else int(rotary_dim)
        code = lib().umim_kv_rollback_rope(ctypes.byref(kv), _p(block_table), max_pages, _p(seq_lens), B,
                                           _p(span_offsets), _p(span_start), _p(span_len), S, _p(surrogate_k),
                                           _p(surrogate_v), _p(rope_inv_freq), rd, _p(freed_pages),
                                           _p(workspace_buf), workspace_buf.numel(), _p(dev_status), _stream(stream))
        _check(code, "umim_kv_rollback_rope")
    return freed_pages


def umim_kv_append(pool, block_table, seq_lens, new_k, new_v, new_pages=None, dev_status=None, stream=None):
    """In-place append of one entry per layer to every sequence (new_k/new_v
    [B][n_layers][Hkv][D] bf16; new_pages [B] int32, read at page boundaries)."""
    kv = paged_kv(pool)
    B, max_pages = block_table.shape
    code = lib().umim_kv_append(ctypes.byref(kv), _p(block_table), max_pages, _p(seq_lens), B, _p(new_k),
                                _p(new_v), _p(new_pages), _p(dev_status), _stream(stream))
    _check(code, "umim_kv_append")


def umim_decode_append_merge(pool, block_table, seq_lens, new_k, new_v, new_pages=None, merge_k=None,
                             merge_row=None, surrogate_k=None, surrogate_v=None, released=None, dev_status=None,
                             stream=None):
    """In place: append new_k/new_v [B][n_layers][Hkv][D] to every sequence,
    or, where merge_k[b] = k > 0, write surrogate row merge_row[b] in place of
    the last k entries (the new one included).  Returns released [B] int32
    (the page a merge freed, or -1)."""
    kv = paged_kv(pool)
    B, max_pages = block_table.shape
    if released is None:
        released = torch.empty(B, dtype=torch.int32, device=pool.device)
    n_rows = 0 if surrogate_k is None else surrogate_k.shape[0]
    code = lib().umim_decode_append_merge(ctypes.byref(kv), _p(block_table), max_pages, _p(seq_lens), B, _p(new_k),
                                          _p(new_v), _p(new_pages), _p(merge_k), _p(merge_row), n_rows,
                                          _p(surrogate_k), _p(surrogate_v), _p(released), _p(dev_status),
                                          _stream(stream))
    _check(code, "umim_decode_append_merge")
    return released


def umim_decode_attention(q, pool, layer, block_table, seq_lens, scale=0.0, out=None, workspace_buf=None,
                          dev_status=None, stream=None):
    """out [B][Hq][D] bf16 = GQA attention of q over the paged cache."""
    dev = _dev(q)
    kv = paged_kv(pool)
    B, Hq, D = q.shape
    max_pages = block_table.shape[1]
    if out is None:
        out = torch.empty_like(q)
    if workspace_buf is None:
        workspace_buf = workspace(umim_decode_attention_workspace_size(B, Hq, kv.n_kv_heads, D), dev)
    code = lib().umim_decode_attention(_p(q), Hq, ctypes.byref(kv), layer, _p(block_table), max_pages,
                                       _p(seq_lens), B, float(scale), _p(out), _p(workspace_buf),
                                       workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_decode_attention")
    return out


def umim_decode_layer_step_workspace_size(batch, n_kv_heads, head_dim):
    return lib().umim_decode_layer_step_workspace_size(batch, n_kv_heads, head_dim)


def umim_decode_layer_step(q, pool, layer, block_table, seq_lens, new_k, new_v, new_pages=None, merge_k=None,
                           merge_row=None, surrogate_k=None, surrogate_v=None, commit=False, released=None,
                           scale=0.0, out=None, workspace_buf=None, dev_status=None, stream=None):
    """One layer of a decode step: writes this layer's new (or, for a merging
    sequence, surrogate) entry and returns out [B][Hq][D] bf16, attention of q
    over the cache with that entry.  new_k / new_v are [B][Hkv][D] views whose
    rows may be strided (e.g. one layer of [B][layers][Hkv][D]); surrogate_k /
    surrogate_v are [rows][Hkv][D].  commit=True on the step's last layer
    records the new lengths, opened pages and released pages.  workspace_buf
    must be zeroed before its first use (workspace() zeroes it)."""
    dev = _dev(q)
    kv = paged_kv(pool)
    B, Hq, D = q.shape
    for t in (new_k, new_v):
        if t.dtype != torch.bfloat16 or t.dim() != 3 or t.shape[0] != B or t.stride(2) != 1 or \
                t.stride(1) != t.shape[2]:
            raise ValueError("new_k / new_v must be bf16 [B][Hkv][D] with contiguous rows")
    if new_k.stride(0) != new_v.stride(0):
        raise ValueError("new_k and new_v must have the same row stride")
    if out is None:
        out = torch.empty_like(q)
    if workspace_buf is None:
        workspace_buf = workspace(umim_decode_layer_step_workspace_size(B, kv.n_kv_heads, D), dev)
    n_rows = 0 if surrogate_k is None else surrogate_k.shape[0]
    code = lib().umim_decode_layer_step(_p(q), Hq, ctypes.byref(kv), layer, _p(block_table), block_table.shape[1],
                                        _p(seq_lens), B, _p(new_k), _p(new_v), new_k.stride(0), _p(new_pages),
                                        _p(merge_k), _p(merge_row), n_rows, _p(surrogate_k), _p(surrogate_v),
                                        1 if commit else 0, _p(released), float(scale), _p(out), _p(workspace_buf),
                                        workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_decode_layer_step")
    return out


def umim_decode_attention_static(q, pool, layer, block_table, seq_lens, scale=0.0, out=None, dev_status=None,
                                 stream=None):
    """Decode attention without a workspace argument, for callers that cannot
    allocate GPU memory at call time: the library's fixed scratch array is
    used instead (see include/umim.h for the size limit and the rule that
    overlapping calls must not run concurrently)."""
    kv = paged_kv(pool)
    B, Hq, D = q.shape
    if out is None:
        out = torch.empty_like(q)
    code = lib().umim_decode_attention_static(_p(q), Hq, ctypes.byref(kv), layer, _p(block_table),
                                              block_table.shape[1], _p(seq_lens), B, float(scale), _p(out),
                                              _p(dev_status), _stream(stream))
    _check(code, "umim_decode_attention_static")
    return out


# ---------------------------------------------------------------------------
# prefill attention and the bounded-wait self-test
# ---------------------------------------------------------------------------
def umim_prefill_attention(q, k, v, cu_seqlens, scale=0.0, out=None, workspace_buf=None, dev_status=None,
                           stream=None):
    """out [T][Hq][D] bf16: causal grouped-query attention within each packed
    sequence of q [T][Hq][D], k / v [T][Hkv][D] (cu_seqlens [B+1] on the device)."""
    dev = _dev(q)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    B = cu_seqlens.numel() - 1
    if out is None:
        out = torch.empty_like(q)
    if workspace_buf is None:
        workspace_buf = workspace(umim_prefill_attention_workspace_size(B, T, Hkv, D), dev)
    code = lib().umim_prefill_attention(_p(q), _p(k), _p(v), T, Hq, Hkv, D, _p(cu_seqlens), B, float(scale), _p(out),
                                        _p(workspace_buf), workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_prefill_attention")
    return out


def umim_selftest_bounded_wait(which, limit_us, device, dev_status=None, stream=None):
    """Run one of the library's bounded waits on something that never happens
    (0: an mbarrier, 1: a counter); returns (status, elapsed_ns)."""
    flags = torch.zeros(2, dtype=torch.int32, device=device)
    elapsed = torch.zeros(1, dtype=torch.int64, device=device)
    status = new_status(device) if dev_status is None else dev_status
    code = lib().umim_selftest_bounded_wait(int(which), int(limit_us), _p(flags), _p(elapsed), _p(status),
                                            _stream(stream))
    _check(code, "umim_selftest_bounded_wait")
    return status, elapsed


def umim_debug_build():
    """1 when the active library is libumim_debug.so, else 0."""
    return int(lib().umim_debug_build())


def umim_debug_site_name(code):
    """The access site named in bits 8.. of a debug build's status word."""
    return lib().umim_debug_site_name(int(code)).decode()


def umim_selftest_bounds_check(buf, index, dev_status=None, stream=None):
    """Debug build only: store 1 into buf[index] (buf a device int32 tensor)
    through the kernels' access-site check; returns the status tensor."""
    status = new_status(buf.device) if dev_status is None else dev_status
    code = lib().umim_selftest_bounds_check(_p(buf), int(buf.numel()), int(index), _p(status), _stream(stream))
    _check(code, "umim_selftest_bounds_check")
    return status


def umim_rule_table_bytes(n_rules):
    return int(lib().umim_rule_table_bytes(n_rules))


def umim_rules_build(rule_tokens, table=None, dev_status=None, stream=None):
    """Rule table for rule_tokens [R][4] int32 (n token ids, then -1s).
    Returns the table (a uint8 device buffer)."""
    R = rule_tokens.shape[0]
    nbytes = umim_rule_table_bytes(R)
    if table is None:
        table = torch.empty(nbytes, dtype=torch.uint8, device=rule_tokens.device)
    code = lib().umim_rules_build(_p(table), table.numel(), _p(rule_tokens), R, _p(dev_status), _stream(stream))
    _check(code, "umim_rules_build")
    return table


def umim_match_prompts_workspace_size(batch, max_len):
    return int(lib().umim_match_prompts_workspace_size(batch, max_len))


def umim_match_prompts(table, token_ids, prompt_lens=None, merge_inputs=False, out=None, workspace_buf=None,
                       dev_status=None, stream=None):
    """Longest-first span selection for a batch of prompts token_ids [B][L].
    Returns (or fills, when out is given) a dict of device int32 tensors:
    span_offsets [B+1], span_start, span_len, span_rule (capacity B*(L//2)),
    and with merge_inputs the span tokens and their CSR offsets
    (merge_token_ids, merge_offsets)."""
    dev = _dev(token_ids)
    B, L = token_ids.shape
    cap = max(1, B * (L // 2))
    i32 = lambda n: torch.empty(n, dtype=torch.int32, device=dev)
    if out is None:
        out = dict(span_offsets=i32(B + 1), span_start=i32(cap), span_len=i32(cap), span_rule=i32(cap),
                   merge_token_ids=i32(max(1, B * L)) if merge_inputs else None,
                   merge_offsets=i32(cap + 1) if merge_inputs else None)
    if workspace_buf is None:
        workspace_buf = workspace(umim_match_prompts_workspace_size(B, L), dev)
    code = lib().umim_match_prompts(_p(table), table.numel(), _p(token_ids), B, L, _p(prompt_lens),
                                    _p(out["span_offsets"]), _p(out["span_start"]), _p(out["span_len"]),
                                    _p(out["span_rule"]), _p(out["merge_token_ids"]), _p(out["merge_offsets"]),
                                    _p(workspace_buf), workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_match_prompts")
    return out


def new_suffix_state(batch, device):
    """Decoding state of umim_match_suffix at the start of generation: [B][4] int32 zeros."""
    return torch.zeros((batch, 4), dtype=torch.int32, device=device)


def umim_match_suffix(table, state, new_tokens, merge_k=None, merge_rule=None, merge_row=None, rows_rule=None,
                      n_merges=None, dev_status=None, stream=None):
    """One decoding step of span selection; state [B][4] is updated in place.
    Returns (merge_k, merge_rule, merge_row, rows_rule, n_merges)."""
    dev = _dev(new_tokens)
    B = new_tokens.shape[0]
    i32 = lambda n: torch.empty(n, dtype=torch.int32, device=dev)
    merge_k = i32(B) if merge_k is None else merge_k
    merge_rule = i32(B) if merge_rule is None else merge_rule
    merge_row = i32(B) if merge_row is None else merge_row
    if rows_rule is None:   # entries past n_merges are not written
        rows_rule = torch.full((max(1, B),), -1, dtype=torch.int32, device=dev)
    n_merges = i32(1) if n_merges is None else n_merges
    code = lib().umim_match_suffix(_p(table), table.numel(), _p(state), _p(new_tokens), B, _p(merge_k),
                                   _p(merge_rule), _p(merge_row), _p(rows_rule), _p(n_merges), _p(dev_status),
                                   _stream(stream))
    _check(code, "umim_match_suffix")
    return merge_k, merge_rule, merge_row, rows_rule, n_merges


def umim_lookup_surrogates(lut, rule_ids, n_dev=None, out=None, dev_status=None, stream=None):
    """out [n][d] fp32 = lut[rule_ids[:n]] with n = min(*n_dev, len(rule_ids))
    (rows past n are left as they were)."""
    R, d = lut.shape
    n_max = rule_ids.shape[0]
    if out is None:
        out = torch.zeros((max(1, n_max), d), dtype=torch.float32, device=lut.device)
    code = lib().umim_lookup_surrogates(_p(lut), R, d, _p(rule_ids), n_max, _p(n_dev), _p(out), _p(dev_status),
                                        _stream(stream))
    _check(code, "umim_lookup_surrogates")
    return out


def umim_distill_align_workspace_size(batch, n_spans):
    return int(lib().umim_distill_align_workspace_size(batch, n_spans))


def umim_distill_align(seq_lens, span_offsets, span_start, span_len, capacity, out=None, workspace_buf=None,
                       dev_status=None, stream=None):
    """Teacher/student row pairs of Algorithm 1 (App. F).  Returns (or fills,
    when out is given) a dict of device int32 tensors: pair_offsets [B+1],
    teacher_rows and student_rows [capacity], student_cu [B+1]."""
    dev = _dev(seq_lens)
    B = seq_lens.numel()
    S = span_start.numel()
    i32 = lambda n: torch.empty(n, dtype=torch.int32, device=dev)
    if out is None:
        out = dict(pair_offsets=i32(B + 1), teacher_rows=i32(max(1, capacity)),
                   student_rows=i32(max(1, capacity)), student_cu=i32(B + 1))
    if workspace_buf is None:
        workspace_buf = workspace(umim_distill_align_workspace_size(B, S), dev)
    code = lib().umim_distill_align(_p(seq_lens), B, _p(span_offsets), _p(span_start), _p(span_len), S,
                                    _p(out["pair_offsets"]), _p(out["teacher_rows"]), _p(out["student_rows"]),
                                    int(capacity), _p(out.get("student_cu")), _p(workspace_buf),
                                    workspace_buf.numel(), _p(dev_status), _stream(stream))
    _check(code, "umim_distill_align")
    return out


def umim_distill_soft_ce_workspace_size(n_student_rows, max_pairs):
    return int(lib().umim_distill_soft_ce_workspace_size(n_student_rows, max_pairs))


def umim_distill_soft_ce(teacher_logits, student_logits, teacher_rows, student_rows, n_pairs=None, vocab=None,
                         eps=1e-8, with_grad=True, loss=None, pair_loss=None, grad=None, workspace_buf=None,
                         dev_status=None, stream=None):
    """Soft-target cross-entropy over the aligned pairs and its gradient with
    respect to the student logits (bf16 [R][ld] rows; vocab defaults to ld).
    n_pairs: device int32 [1] (pairs used: its value) or None (all of
    teacher_rows).  Returns (loss [1] fp32, pair_loss [max_pairs] fp32,
    grad bf16 like student_logits or None)."""
    dev = _dev(student_logits)
    R_T, ld = teacher_logits.shape
    R_S = student_logits.shape[0]
    if student_logits.shape[1] != ld or teacher_logits.dtype != torch.bfloat16 or \
            student_logits.dtype != torch.bfloat16:
        raise ValueError("logits must be bf16 [rows][ld] with the same ld")
    V = ld if vocab is None else int(vocab)
    P = teacher_rows.numel()
    if loss is None:
        loss = torch.empty(1, dtype=torch.float32, device=dev)
    if pair_loss is None:
        pair_loss = torch.empty(max(1, P), dtype=torch.float32, device=dev)
    if with_grad and grad is None:
        grad = torch.empty_like(student_logits)
    if workspace_buf is None:
        workspace_buf = workspace(umim_distill_soft_ce_workspace_size(R_S, P), dev)
    code = lib().umim_distill_soft_ce(_p(teacher_logits), R_T, _p(student_logits), R_S, V, ld, _p(teacher_rows),
                                      _p(student_rows), P, _p(n_pairs), float(eps), _p(loss), _p(pair_loss),
                                      _p(grad if with_grad else None), _p(workspace_buf), workspace_buf.numel(),
                                      _p(dev_status), _stream(stream))
    _check(code, "umim_distill_soft_ce")
    return loss, pair_loss, (grad if with_grad else None)


# ---------------------------------------------------------------------------
# kernel tracing (profiling aid)
# ---------------------------------------------------------------------------
def trace_start(capacity=4096):
    _check(lib().umim_trace_start(capacity), "umim_trace_start")


def trace_stop():
    lib().umim_trace_stop()


def trace_read(cap=4096):
    """[(label, milliseconds)] of every kernel launched while tracing."""
    ms = (ctypes.c_float * cap)()
    labels = (ctypes.c_char_p * cap)()
    n = lib().umim_trace_read(ms, labels, cap)
    return [(labels[i].decode(), float(ms[i])) for i in range(n)]
