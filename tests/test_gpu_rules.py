"""Merge-rule matching and the surrogate lookup on the GPU against the oracle
(App. E "Rule Matching", "Prompt Merging", "Decoding-Time Merging").

Bit-exact throughout: span lists, rule ids and merge-module inputs of prompt
matching; merge lengths, rows, rule ids and the per-sequence state of every
decoding step; looked-up surrogate rows.  End to end, prompt compression with
looked-up surrogates equals prompt compression with the merge module run on
the matched spans, and a decode loop driven by the GPU suffix matcher leaves
the cache exactly where the oracle's does.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import rules as OR
import workloads as W
from helpers import dev, oracle_append_merge, umim

pytestmark = pytest.mark.gpu


def _rules_np(tuples):
    r = np.full((len(tuples), 4), -1, np.int32)
    for i, g in enumerate(tuples):
        r[i, :len(g)] = g
    return r


def _small_rules(seed, vocab, n):
    r = W.rng(seed)
    out = set()
    while len(out) < n:
        k = int(r.integers(2, 5))
        out.add(tuple(int(x) for x in r.integers(0, vocab, size=k)))
    return sorted(out, key=lambda g: (len(g), g))


def _build(m, rules, dv):
    status = m.new_status(dv)
    table = m.umim_rules_build(torch.from_numpy(rules).to(dv), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return table


def _check_prompts(out, toks, lens, rules_d, merge_inputs):
    offs, st, ln, rl = OR.match_prompts(toks, lens, rules_d)
    g_offs = out["span_offsets"].cpu().numpy()
    np.testing.assert_array_equal(g_offs, offs)
    S = int(offs[-1])
    np.testing.assert_array_equal(out["span_start"][:S].cpu().numpy(), st)
    np.testing.assert_array_equal(out["span_len"][:S].cpu().numpy(), ln)
    np.testing.assert_array_equal(out["span_rule"][:S].cpu().numpy(), rl)
    if merge_inputs:
        want_t, want_o = [], [0]
        for b in range(len(lens)):
            for j in range(offs[b], offs[b + 1]):
                want_t += list(toks[b][st[j]:st[j] + ln[j]])
                want_o.append(len(want_t))
        np.testing.assert_array_equal(out["merge_offsets"][:S + 1].cpu().numpy(), want_o)
        np.testing.assert_array_equal(out["merge_token_ids"][:len(want_t)].cpu().numpy(), want_t)
    return S


@pytest.mark.parametrize("seed,vocab,n_rules,lens,L,coverage", [
    # dense matches over a tiny alphabet; prompts across the 2048-position passes
    (51, 5, 60, [0, 1, 2, 3, 17, 2047, 2048, 2049, 4500], 4500, None),
    # planted rules in a large vocabulary, ragged lengths
    (52, 50000, 5000, [3000, 2999, 1, 0, 1500, 2048, 4, 777, 3000, 2100, 5, 6, 7, 8, 9, 2500], 3000, 0.4),
    # one prompt, every 2-gram of a 2-symbol alphabet and every 3-gram a rule
    (53, 2, 12, [4097], 4097, None),
])
def test_prompt_matching_matches_oracle(seed, vocab, n_rules, lens, L, coverage):
    m, dv = umim(), dev()
    if seed == 53:
        tuples = [(a, b) for a in range(2) for b in range(2)] + \
                 [(a, b, c) for a in range(2) for b in range(2) for c in range(2)]
    else:
        tuples = _small_rules(seed, vocab, n_rules)
    rules = _rules_np(tuples)
    if coverage is None:
        toks = W.rng(seed + 1).integers(0, vocab, size=(len(lens), L)).astype(np.int32)
    else:
        toks = W.rule_prompts(seed + 1, rules, B=len(lens), L=L, vocab=vocab, coverage=coverage, lens=lens)
    table = _build(m, rules, dv)
    status = m.new_status(dv)
    for merge_inputs in (False, True):
        out = m.umim_match_prompts(table, torch.from_numpy(toks).to(dv), torch.tensor(lens, dtype=torch.int32,
                                   device=dv), merge_inputs=merge_inputs, dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        S = _check_prompts(out, toks, lens, OR.rule_dict(tuples), merge_inputs)
    assert S > 0


def test_prompt_matching_full_rule_set():
    """The Llama-3 rule set (2.2 million rules) over 64 prompts of 2048 tokens
    with 40 % of each covered by planted rules (the prompt-compression shape)."""
    m, dv = umim(), dev()
    rules = W.random_rules(W.SEEDS["rule_matching"], W.LLAMA3_RULE_COUNTS, W.LLAMA3_VOCAB)
    toks = W.rule_prompts(W.SEEDS["rule_matching"] + 1, rules, B=64, L=2048, vocab=W.LLAMA3_VOCAB, coverage=0.4)
    table = _build(m, rules, dv)
    status = m.new_status(dv)
    out = m.umim_match_prompts(table, torch.from_numpy(toks).to(dv), merge_inputs=True, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    S = _check_prompts(out, toks, [2048] * 64, OR.rule_dict(W.rule_tuples(rules)), True)
    assert 0.35 < S * 3 / toks.size < 0.45


def test_invalid_rules_and_tokens_are_reported():
    m, dv = umim(), dev()
    # a repeated n-gram
    status = m.new_status(dv)
    m.umim_rules_build(torch.from_numpy(_rules_np([(1, 2), (3, 4, 5), (1, 2)])).to(dv), dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1
    # malformed rows: one token; a gap; a token id past 24 bits
    for bad in ([[7, -1, -1, -1]], [[1, -1, 2, -1]], [[1, 1 << 24, -1, -1]]):
        status = m.new_status(dv)
        m.umim_rules_build(torch.tensor(bad, dtype=torch.int32, device=dv), dev_status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 1
    # prompt tokens outside the id range match nothing and are reported
    table = _build(m, _rules_np([(1, 2), (2, 3)]), dv)
    toks = torch.tensor([[1, 2, -5, 2, 3, 1, 2]], dtype=torch.int32, device=dv)
    status = m.new_status(dv)
    out = m.umim_match_prompts(table, toks, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1
    assert out["span_offsets"].cpu().tolist() == [0, 3]
    assert out["span_start"][:3].cpu().tolist() == [0, 3, 5]
    # the table must be large enough
    with pytest.raises(m.UmimError):
        m.umim_rules_build(torch.from_numpy(_rules_np(_small_rules(1, 100, 20))).to(dv),
                           table=torch.empty(256, dtype=torch.uint8, device=dv))


@pytest.mark.parametrize("seed,vocab,n_rules,B,steps", [
    (61, 4, 30, 37, 300),
    (62, 6, 80, 1100, 40),     # more sequences than one pass of the kernel's block
])
def test_suffix_matching_every_step(seed, vocab, n_rules, B, steps):
    m, dv = umim(), dev()
    tuples = _small_rules(seed, vocab, n_rules)
    rules_d = OR.rule_dict(tuples)
    table = _build(m, _rules_np(tuples), dv)
    state = m.new_suffix_state(B, dv)
    states = [OR.SuffixState() for _ in range(B)]
    status = m.new_status(dv)
    r = W.rng(seed + 5)
    total = 0
    for step in range(steps):
        y = r.integers(0, vocab, size=B).astype(np.int32)
        k, rule, row, rows_rule, n = m.umim_match_suffix(table, state, torch.from_numpy(y).to(dv),
                                                         dev_status=status)
        wk, wr, wrow, wrows = OR.match_suffixes(states, y, rules_d)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        np.testing.assert_array_equal(k.cpu().numpy(), wk, err_msg=f"step {step}")
        np.testing.assert_array_equal(rule.cpu().numpy(), wr, err_msg=f"step {step}")
        np.testing.assert_array_equal(row.cpu().numpy(), wrow, err_msg=f"step {step}")
        assert int(n.item()) == len(wrows)
        np.testing.assert_array_equal(rows_rule[:len(wrows)].cpu().numpy(), wrows)
        st = state.cpu().numpy()
        for b in range(B):
            nr = int(st[b, 3])
            assert nr == len(states[b].raw) and list(st[b, 3 - nr:3]) == states[b].raw, (step, b)
        total += len(wrows)
    assert total > 0


def test_lookup_matches_indexing():
    m, dv = umim(), dev()
    g = torch.Generator(device=dv)
    g.manual_seed(71)
    lut = torch.randn((1000, 64), generator=g, device=dv)
    ids = torch.randint(0, 1000, (300,), generator=g, device=dv, dtype=torch.int32)
    n_dev = torch.tensor([217], dtype=torch.int32, device=dv)
    status = m.new_status(dv)
    out = m.umim_lookup_surrogates(lut, ids, n_dev=n_dev, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    want = OR.lookup(lut.cpu().numpy(), ids.cpu().numpy()[:217])
    np.testing.assert_array_equal(out[:217].cpu().numpy(), want)
    assert torch.all(out[217:] == 0)
    bad = torch.tensor([3, 1000, -1], dtype=torch.int32, device=dv)
    out = m.umim_lookup_surrogates(lut, bad, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 1
    np.testing.assert_array_equal(out[0].cpu().numpy(), lut[3].cpu().numpy())
    assert torch.all(out[1:] == 0)


def test_prompt_compression_with_lookup_equals_merge_module():
    """Surrogates precomputed once per rule by the merge module and fetched by
    rule id give, bit for bit, the compressed prompts that running the merge
    module on the matched spans gives."""
    m, dv = umim(), dev()
    vocab, d, h = 3000, 512, 4
    tuples = _small_rules(81, vocab, 400)
    rules = _rules_np(tuples)
    B, L = 6, 700
    lens = [L] * B
    toks = W.rule_prompts(82, rules, B=B, L=L, vocab=vocab, coverage=0.4)
    emb = W.bf16_normal((vocab, d), 0.02, 83, dv)
    w = W.merge_weights(d, h, 84, dv)
    table = _build(m, rules, dv)
    status = m.new_status(dv)
    # the lookup table: the merge module over every rule's n-gram
    flat = torch.from_numpy(np.concatenate([np.asarray(g, np.int32) for g in tuples])).to(dv)
    offs = torch.from_numpy(np.concatenate([[0], np.cumsum([len(g) for g in tuples])]).astype(np.int32)).to(dv)
    lut = m.umim_merge_spans(emb, flat, offs, w, dev_status=status)
    t_toks = torch.from_numpy(toks).to(dv)
    out = m.umim_match_prompts(table, t_toks, merge_inputs=True, dev_status=status)
    torch.cuda.synchronize()
    S = _check_prompts(out, toks, lens, OR.rule_dict(tuples), True)
    assert S > 50
    # path 1: fetch by rule id (device-side count)
    sur_lut = m.umim_lookup_surrogates(lut, out["span_rule"], n_dev=out["span_offsets"][B:], dev_status=status)
    # path 2: the merge module on the matched spans
    T = int(out["merge_offsets"][S].item())
    sur_mm = m.umim_merge_spans(emb, out["merge_token_ids"][:T], out["merge_offsets"][:S + 1], w, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(sur_lut[:S], sur_mm)
    c1 = m.umim_build_compressed(emb, t_toks, out["span_offsets"], out["span_start"], out["span_len"], sur_lut,
                                 dev_status=status)
    c2 = m.umim_build_compressed(emb, t_toks, out["span_offsets"], out["span_start"], out["span_len"], sur_mm,
                                 dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    rows = int(c1[2][-1].item())
    assert rows == B * L - sum(int(x) - 1 for x in out["span_len"][:S].cpu().tolist())
    assert torch.equal(c1[0][:rows], c2[0][:rows])
    assert torch.equal(c1[1][:rows], c2[1][:rows]) and torch.equal(c1[2], c2[2])


def test_decode_loop_driven_by_the_suffix_matcher():
    """Each step: the GPU suffix matcher decides, per sequence, between an
    append and a merge of the last n entries; umim_decode_append_merge applies
    it with per-rule surrogate KV rows.  The cache, block tables and lengths
    follow the oracle (SuffixState, then append and suffix rollback)."""
    m, dv = umim(), dev()
    vocab, B, layers, hkv, hd, steps = 5, 9, 2, 2, 64, 60
    tuples = _small_rules(91, vocab, 25)
    rules_d = OR.rule_dict(tuples)
    table = _build(m, _rules_np(tuples), dv)
    lens = [5, 16, 31, 100, 1, 47, 64, 15, 200]
    extra = steps // 16 + 2
    c = W.decode_case(92, lens=lens, n_q_heads=hkv, n_kv_heads=hkv, head_dim=hd, n_layers=layers, coverage=0.0,
                      spare_pages=B * extra, extra_max_pages=extra)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    o_pool, o_bt, o_lens = W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy()
    used = set(int(x) for x in o_bt[o_bt >= 0].ravel())
    alloc = W.PageAllocator([p for p in range(c.n_pages) if p not in used])
    # one surrogate KV row per rule (stands in for the backbone's forward of the surrogate)
    kv_lut_k = W.bf16_normal((len(tuples), layers, hkv, hd), 1.0, 93, dv)
    kv_lut_v = W.bf16_normal((len(tuples), layers, hkv, hd), 1.0, 94, dv)
    state = m.new_suffix_state(B, dv)
    states = [OR.SuffixState() for _ in range(B)]
    status = m.new_status(dv)
    r = W.rng(95)
    n_merges = 0
    for step in range(steps):
        y = r.integers(0, vocab, size=B).astype(np.int32)
        nk = W.bf16_normal((B, layers, hkv, hd), 1.0, 9000 + 2 * step, dv)
        nv = W.bf16_normal((B, layers, hkv, hd), 1.0, 9001 + 2 * step, dv)
        new_pages = alloc.take(o_lens)
        k, rule, row, rows_rule, n = m.umim_match_suffix(table, state, torch.from_numpy(y).to(dv),
                                                         dev_status=status)
        # only the first n entries of rows_rule are written
        n_rows = int(n.item())
        idx = rows_rule[:n_rows].long()
        sk, sv = (kv_lut_k[idx], kv_lut_v[idx]) if n_rows else (None, None)
        rel = m.umim_decode_append_merge(pool, bt, sl, nk, nv, torch.from_numpy(new_pages).to(dv), k, row, sk, sv,
                                         dev_status=status)
        wk, wr, wrow, wrows = OR.match_suffixes(states, y, rules_d)
        o_pool, o_bt, o_lens, o_rel = oracle_append_merge(o_pool, o_bt, o_lens, W.bits(nk), W.bits(nv), new_pages,
                                                          wk, W.bits(kv_lut_k)[wrows], W.bits(kv_lut_v)[wrows])
        alloc.give_back([p for p in o_rel if p >= 0])
        n_merges += len(wrows)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        np.testing.assert_array_equal(k.cpu().numpy(), wk)
        np.testing.assert_array_equal(bt.cpu().numpy(), o_bt, err_msg=f"step {step}")
        np.testing.assert_array_equal(sl.cpu().numpy(), o_lens, err_msg=f"step {step}")
        np.testing.assert_array_equal(rel.cpu().numpy(), o_rel, err_msg=f"step {step}")
    gp = W.bits(pool)
    for b in range(B):
        t = np.arange(int(o_lens[b]))
        pg, slot = o_bt[b, t // 16], t % 16
        np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], o_pool[:, pg, :, :, slot, :], err_msg=f"seq {b}")
    assert n_merges > 0
