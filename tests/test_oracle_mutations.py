"""Planted mistakes in the oracle are caught by its pins (CPU only).

Each case swaps one piece of the oracle for a plausible slip (a transposed
weight, the wrong softmax scale, an unbiased variance, swapped K and V, a
page released one too few, ...), runs the pins of that function from
tests/test_oracle_*.py, and checks that at least one of them fails.  The
mistakes live only in this file, are planted in the oracle on the CPU, and
are undone after each case; the unmodified oracle passes every pin (the pin
files themselves check that).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import append as AP
from oracle import attention as A
from oracle import distill as D
from oracle import merge as M
from oracle import rollback as R
import test_oracle_append as TAP
import test_oracle_attention as TA
import test_oracle_compaction as TC
import test_oracle_distill as TD
import test_oracle_merge as TM
import test_oracle_prefill as TP
import test_oracle_rollback as TR
from oracle import bf16 as OB
from oracle import compaction as C


def _failures(pins):
    """How many pins fail: an assertion, or the oracle's own input checks
    refusing the state the planted mistake left behind."""
    n = 0
    for fn, args in pins:
        try:
            fn(*args)
        except (AssertionError, ValueError):
            n += 1
    return n


# ---------------------------------------------------------------------------
# merge module (App. C.1)
# ---------------------------------------------------------------------------
MERGE_PINS = [
    (TM.test_single_token_span_is_library_chain, (64, 4)),
    (TM.test_single_token_span_is_library_chain, (256, 8)),
    (TM.test_pooling_is_library_sdpa, ()),
    (TM.test_repeated_token_equals_single_token, ()),
    (TM.test_token_order_does_not_matter, ()),
    (TM.test_zero_query_is_mean_pooling, ()),
    (TM.test_brute_force_tiny, ()),
    (TM.test_listing_semantics_batched, ()),
    (TM.test_gelu_is_erf_form, ()),
]


def _pool(strided=False, scale_full_width=False, normalise=True):
    def attention_pool(P, q, n_heads):
        n, d = P.shape
        dh = d // n_heads
        o = np.empty(d)
        alphas = np.empty((n_heads, n))
        for i in range(n_heads):
            cols = np.arange(i, d, n_heads) if strided else np.arange(i * dh, (i + 1) * dh)
            Pi = P[:, cols]
            s = Pi @ q[i] / math.sqrt(d if scale_full_width else dh)
            e = np.exp(s - s.max())
            a = e / e.sum() if normalise else e
            alphas[i] = a
            o[cols] = a @ Pi
        return o, alphas
    return attention_pool


def _ln(ddof=0, affine=True, eps_inside=True):
    def layer_norm(x, gamma, beta, eps):
        mu = x.mean(axis=-1, keepdims=True)
        var = x.var(axis=-1, keepdims=True, ddof=ddof)
        y = (x - mu) / (np.sqrt(var + eps) if eps_inside else np.sqrt(var) + eps)
        return y * gamma + beta if affine else y
    return layer_norm


MERGE_MUTATIONS = {
    "weight used untransposed": {"linear": lambda x, w, b: x @ w + b},
    "bias dropped": {"linear": lambda x, w, b: x @ w.T},
    "tanh GELU": {"gelu": lambda x: 0.5 * x * (1 + np.tanh(math.sqrt(2 / math.pi) * (x + 0.044715 * x ** 3)))},
    "unbiased variance": {"layer_norm": _ln(ddof=1)},
    "LayerNorm without gamma / beta": {"layer_norm": _ln(affine=False)},
    "eps outside the square root": {"layer_norm": _ln(eps_inside=False)},
    "scores scaled by sqrt(d) instead of sqrt(d_h)": {"attention_pool": _pool(scale_full_width=True)},
    "heads taken as strided columns": {"attention_pool": _pool(strided=True)},
    "unnormalised pooling weights": {"attention_pool": _pool(normalise=False)},
    "GELU missing after the output projection": {
        "output_processor": lambda o, w, eps: M.layer_norm(M.linear(o, w["w_o"], w["b_o"]), w["ln_o_gamma"],
                                                           w["ln_o_beta"], eps)},
}


@pytest.mark.parametrize("name", sorted(MERGE_MUTATIONS))
def test_merge_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        for attr, fn in MERGE_MUTATIONS[name].items():
            mp.setattr(M, attr, fn)
        assert _failures(MERGE_PINS) >= 1, name


# ---------------------------------------------------------------------------
# decode attention
# ---------------------------------------------------------------------------
ATTENTION_PINS = [
    (TA.test_matches_library_sdpa_gqa, (8, 2, 64)),
    (TA.test_matches_library_sdpa_gqa, (4, 4, 16)),
    (TA.test_closed_forms, ()),
    (TA.test_empty_cache_gives_zero, ()),
    (TA.test_after_rollback_equals_rebuilt_cache, ()),
]
_attend = A.attend
_decode = A.decode_attention


def _interleaved_heads(q_bits, pool_bits, layer, block_table, seq_lens, **kw):
    """Query head h read KV head h mod Hkv instead of h // G."""
    Hq, Hkv = q_bits.shape[1], pool_bits.shape[3]
    G = Hq // Hkv
    perm = np.array([(h % Hkv) * G + h // Hkv for h in range(Hq)])
    q2 = np.empty_like(q_bits)
    q2[:, perm] = q_bits
    res = _decode(q2, pool_bits, layer, block_table, seq_lens, **kw)
    if kw.get("return_weights"):
        out, w = res
        return out[:, perm], [[wb[p] for p in perm] for wb in w]
    return res[:, perm]


ATTENTION_MUTATIONS = {
    "scale 1/D": {"attend": lambda q, K, V, s: _attend(q, K, V, s * s)},
    "K and V swapped": {"attend": lambda q, K, V, s: _attend(q, V, K, s)},
    "last entry left out": {"attend": lambda q, K, V, s: _attend(q, K[:-1], V[:-1], s) if len(K) > 1
                            else _attend(q, K, V, s)},
    "grouped heads interleaved": {"decode_attention": _interleaved_heads},
}


@pytest.mark.parametrize("name", sorted(ATTENTION_MUTATIONS))
def test_attention_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        for attr, fn in ATTENTION_MUTATIONS[name].items():
            mp.setattr(A, attr, fn)
            if attr == "decode_attention":
                mp.setattr(oracle, attr, fn)
        assert _failures(ATTENTION_PINS) >= 1, name


# ---------------------------------------------------------------------------
# KV rollback (App. E, App. C.6)
# ---------------------------------------------------------------------------
ROLLBACK_PINS = [
    (TR.test_worked_example_app_c5, ()),
    (TR.test_decode_cache_length_formula, ()),
    (TR.test_length_formula_many_spans, ()),
    (TR.test_k1_with_stored_entry_is_identity, ()),
    (TR.test_against_list_brute_force, (5, [512], 1, 0.4)),
    (TR.test_against_list_brute_force, (6, [100, 0, 17, 300, 16, 32], 2, 0.3)),
    (TR.test_untouched_prefix_and_freed_pages, ()),
    (TR.test_page_aligned_lengths, (20, [(0, 5)], 16, 1)),
    (TR.test_page_aligned_lengths, (33, [(1, 2)], 32, 2)),
]
_rollback = R.kv_rollback


def _surrogates_swapped(pool, bt, lens, offs, st, ln, sk, sv, **kw):
    return _rollback(pool, bt, lens, offs, st, ln, sv, sk, **kw)


def _one_page_too_few_released(pool, bt, lens, offs, st, ln, sk, sv, **kw):
    p2, bt2, l2, freed = _rollback(pool, bt, lens, offs, st, ln, sk, sv, **kw)
    if freed:
        b, i = np.argwhere(np.asarray(bt) == freed[-1])[0]
        bt2[b, i] = freed[-1]
        freed = freed[:-1]
    return p2, bt2, l2, freed


def _length_minus_k(pool, bt, lens, offs, st, ln, sk, sv, **kw):
    p2, bt2, l2, freed = _rollback(pool, bt, lens, offs, st, ln, sk, sv, **kw)
    return p2, bt2, l2 - np.diff(np.asarray(offs)).astype(l2.dtype), freed


def _spans_one_by_one_unadjusted(pool, bt, lens, offs, st, ln, sk, sv, **kw):
    """Each span applied on its own, left to right, at its original start
    (the starts of later spans not moved by the earlier removals; a span that
    no longer fits is skipped, so only the pins can tell)."""
    offs = np.asarray(offs)
    B = len(lens)
    freed_all = []
    for b in range(B):
        for i in range(int(offs[b]), int(offs[b + 1])):
            if int(st[i]) + int(ln[i]) > int(np.asarray(lens)[b]):
                continue
            o = np.zeros(B + 1, np.int32)
            o[b + 1:] = 1
            pool, bt, lens, freed = _rollback(pool, bt, lens, o, np.asarray(st)[i:i + 1], np.asarray(ln)[i:i + 1],
                                              np.asarray(sk)[i:i + 1], np.asarray(sv)[i:i + 1], **kw)
            freed_all += freed
    return pool, bt, lens, freed_all


ROLLBACK_MUTATIONS = {
    "surrogate K and V swapped": _surrogates_swapped,
    "one page too few released": _one_page_too_few_released,
    "length L - sum k instead of L - sum (k - 1)": _length_minus_k,
    "spans applied one by one at unadjusted starts": _spans_one_by_one_unadjusted,
}


@pytest.mark.parametrize("name", sorted(ROLLBACK_MUTATIONS))
def test_rollback_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        mp.setattr(R, "kv_rollback", ROLLBACK_MUTATIONS[name])
        mp.setattr(oracle, "kv_rollback", ROLLBACK_MUTATIONS[name])
        assert _failures(ROLLBACK_PINS) >= 1, name


# ---------------------------------------------------------------------------
# aligned predictive distillation (App. F, Algorithm 1)
# ---------------------------------------------------------------------------
DISTILL_PINS = [
    (TD.test_paper_alignment_example, ()),
    (TD.test_packed_pairs_follow_the_compressed_position_map, (0,)),
    (TD.test_packed_pairs_follow_the_compressed_position_map, (3,)),
    (TD.test_loss_is_library_soft_cross_entropy_and_kl, ()),
    (TD.test_gradient_matches_autograd, (0.0,)),
    (TD.test_gradient_matches_autograd, (1e-3,)),
    (TD.test_no_spans_no_pairs_and_zero_loss, ()),
]


def _soft_ce_variant(drop_eps_in_grad=False, no_mean=False):
    def soft_ce(teacher_logits, student_logits, teacher_rows, student_rows, eps=1e-8):
        N = len(teacher_rows)
        grad = np.zeros(np.shape(student_logits))
        if N == 0:
            return 0.0, grad
        total = 0.0
        for t, s in zip(teacher_rows, student_rows):
            pt = D._softmax(np.asarray(teacher_logits[t], dtype=np.float64))
            ps = D._softmax(np.asarray(student_logits[s], dtype=np.float64))
            total += float(np.sum(pt * np.log(ps + eps)))
            a = pt if drop_eps_in_grad else pt * ps / (ps + eps)
            grad[s] += -(a - ps * a.sum()) / (1 if no_mean else N)
        return -total / (1 if no_mean else N), grad
    return soft_ce


def _align_anchor_first(lens, span_offsets, span_start, span_len):
    """The surrogate paired with the span's first position instead of its last."""
    offs, tpos, spos = [0], [], []
    for b in range(len(lens)):
        L = int(lens[b])
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        if hi == lo:
            offs.append(len(tpos))
            continue
        keep = np.ones(L, bool)
        removed = 0
        for i in range(lo, hi):
            s, n = int(span_start[i]), int(span_len[i])
            keep[s + 1:s + n] = False
            removed += n - 1
        first = int(span_start[lo])
        teacher = [j for j in range(L) if keep[j] and j >= first]
        Lc = L - removed
        tpos += teacher
        spos += list(range(Lc - len(teacher), Lc))
        offs.append(len(tpos))
    return tuple(np.asarray(x, dtype=np.int32) for x in (offs, tpos, spos))


DISTILL_MUTATIONS = {
    "gradient without the eps term": {"soft_ce": _soft_ce_variant(drop_eps_in_grad=True)},
    "sum over pairs instead of the mean": {"soft_ce": _soft_ce_variant(no_mean=True)},
    "surrogate aligned with the span's first position": {"align": _align_anchor_first},
}


@pytest.mark.parametrize("name", sorted(DISTILL_MUTATIONS))
def test_distill_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        for attr, fn in DISTILL_MUTATIONS[name].items():
            mp.setattr(D, attr, fn)
            mp.setattr(TD, attr, fn)
        assert _failures(DISTILL_PINS) >= 1, name


# ---------------------------------------------------------------------------
# compressed prompts (App. C.5, App. E "Prompt Merging", App. J.4)
# ---------------------------------------------------------------------------
COMPACTION_PINS = [
    (TC.test_worked_example, ()),
    (TC.test_compressed_length_formula, ()),
    (TC.test_no_spans_is_embedding_lookup, ()),
    (TC.test_bf16_rounding_matches_torch, ()),
]
_build = C.build_compressed


def _positions_kept_from_the_original(table_bits, token_ids, span_offsets, span_start, span_len, surrogates):
    """Position ids that keep each unit's original index (t) instead of
    renumbering the compressed sequence 0 .. L'-1."""
    out, pos, cu = _build(table_bits, token_ids, span_offsets, span_start, span_len, surrogates)
    B, L = np.asarray(token_ids).shape
    orig = []
    for b in range(B):
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        t, i = 0, lo
        while t < L:
            orig.append(t)
            if i < hi and t == int(span_start[i]):
                t += int(span_len[i])
                i += 1
            else:
                t += 1
    return out, np.asarray(orig, np.int32), cu


class _TruncatingBf16:
    """bf16 conversions with the rounding replaced by truncation."""
    to_f64 = staticmethod(OB.to_f64)

    @staticmethod
    def from_f32(x):
        return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)

    from_f64 = staticmethod(OB.from_f64)


COMPACTION_MUTATIONS = {
    "original positions kept": ("build_compressed", _positions_kept_from_the_original),
    "surrogates rounded to bf16 by truncation": ("bf16", _TruncatingBf16),
}


@pytest.mark.parametrize("name", sorted(COMPACTION_MUTATIONS))
def test_compaction_pins_catch(name):
    attr, fn = COMPACTION_MUTATIONS[name]
    with pytest.MonkeyPatch.context() as mp:
        mp.setattr(C, attr, fn)
        if attr == "build_compressed":
            mp.setattr(oracle, attr, fn)
        else:   # the pins convert through the same module
            mp.setattr(TC, "bf16", fn)
        assert _failures(COMPACTION_PINS) >= 1, name


# ---------------------------------------------------------------------------
# prefill attention over packed compressed prompts
# ---------------------------------------------------------------------------
PREFILL_PINS = [
    (TP.test_matches_library_causal_sdpa, (8, 2, 32)),
    (TP.test_closed_forms, ()),
    (TP.test_packing_is_per_sequence, ()),
    (TP.test_last_row_is_decode_attention, ()),
]


def _prefill_variant(keys_to=lambda lo, hi, i: i + 1, first_key=lambda lo, i: lo):
    def prefill_attention(q_bits, k_bits, v_bits, cu_seqlens, scale=None, rows=None):
        q, k, v = OB.to_f64(q_bits), OB.to_f64(k_bits), OB.to_f64(v_bits)
        T, Hq, D = q.shape
        G = Hq // k.shape[1]
        scale = 1.0 / math.sqrt(D) if not scale else scale
        cu = np.asarray(cu_seqlens)
        out = np.zeros((T, Hq, D))
        for b in range(len(cu) - 1):
            lo, hi = int(cu[b]), int(cu[b + 1])
            for i in range(lo, hi):
                a, z = first_key(lo, i), keys_to(lo, hi, i)
                if z <= a:
                    continue
                for h in range(Hq):
                    s = (k[a:z, h // G, :] @ q[i, h]) * scale
                    e = np.exp(s - s.max())
                    out[i, h] = (e / e.sum()) @ v[a:z, h // G, :]
        return out
    return prefill_attention


PREFILL_MUTATIONS = {
    "no causal mask": _prefill_variant(keys_to=lambda lo, hi, i: hi),
    "diagonal masked out": _prefill_variant(keys_to=lambda lo, hi, i: i if i > lo else i + 1),
    "keys of earlier sequences visible": _prefill_variant(first_key=lambda lo, i: 0),
}


@pytest.mark.parametrize("name", sorted(PREFILL_MUTATIONS))
def test_prefill_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        mp.setattr(TP, "prefill_attention", PREFILL_MUTATIONS[name])
        assert _failures(PREFILL_PINS) >= 1, name


# ---------------------------------------------------------------------------
# decode-step append (App. E, Fig. 2 step (2))
# ---------------------------------------------------------------------------
APPEND_PINS = [
    (TAP.test_append_matches_logical_list_model, ()),
    (TAP.test_page_opened_only_at_boundary, ()),
    (TAP.test_append_then_replace_by_one_entry_is_appending_that_entry, ()),
    (TAP.test_appending_n_then_merging_them_is_appending_the_surrogate, (3,)),
    (TAP.test_appending_n_then_merging_them_is_appending_the_surrogate, (17,)),
    (TAP.test_rejected_sequences_are_left_unchanged, ()),
]
_append = AP.kv_append


def _append_variant(slot_shift=0, page_every_call=False, k_into_v=False):
    def kv_append(pool, block_table, seq_lens, new_k, new_v, new_pages=None, page_size=16):
        P = page_size
        pool = np.array(pool, copy=True)
        bt = np.array(block_table, dtype=np.int32, copy=True)
        lens = np.array(seq_lens, dtype=np.int32, copy=True)
        rejected = []
        for b in range(bt.shape[0]):
            L = int(lens[b])
            t = L + slot_shift
            if L < 0 or t >= bt.shape[1] * P:
                rejected.append(b)
                continue
            opens = page_every_call or t % P == 0
            page = (-1 if new_pages is None else int(new_pages[b])) if opens else int(bt[b, t // P])
            if page < 0 or page >= pool.shape[1]:
                rejected.append(b)
                continue
            bt[b, t // P] = page
            pool[:, page, 0, :, t % P, :] = new_k[b]
            pool[:, page, 1, :, t % P, :] = new_k[b] if k_into_v else new_v[b]
            lens[b] = L + 1
        return pool, bt, lens, rejected
    return kv_append


APPEND_MUTATIONS = {
    "written one slot too far": _append_variant(slot_shift=1),
    "a new page taken on every append": _append_variant(page_every_call=True),
    "K written into the V slot too": _append_variant(k_into_v=True),
}


@pytest.mark.parametrize("name", sorted(APPEND_MUTATIONS))
def test_append_pins_catch(name):
    with pytest.MonkeyPatch.context() as mp:
        mp.setattr(AP, "kv_append", APPEND_MUTATIONS[name])
        mp.setattr(oracle, "kv_append", APPEND_MUTATIONS[name])
        assert _failures(APPEND_PINS) >= 1, name


def test_unmodified_oracle_passes_the_same_pins():
    assert _failures(MERGE_PINS + ATTENTION_PINS + ROLLBACK_PINS + DISTILL_PINS + COMPACTION_PINS +
                     PREFILL_PINS + APPEND_PINS) == 0
