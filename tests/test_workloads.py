"""The seeded input generators follow the stated recipe: spans sorted,
non-overlapping, of lengths kmin..kmax and covering the requested fraction;
physical pages a permutation of the pool; serving lengths lognormal and
clipped; distinct rules planted over about the requested fraction of each
prompt; every draw reproducible from its seed.  CPU only."""
import numpy as np
import pytest
import torch

import workloads as W


def _check_spans(st, ln, L, kmin, kmax):
    assert st.dtype == np.int32 and ln.dtype == np.int32 and len(st) == len(ln)
    if len(st) == 0:
        return
    assert np.all((ln >= kmin) & (ln <= kmax))
    assert st[0] >= 0 and st[-1] + ln[-1] <= L
    assert np.all(st[1:] >= st[:-1] + ln[:-1])      # sorted, non-overlapping


@pytest.mark.parametrize("L,cov,kmin,kmax", [(4096, 0.3, 2, 4), (32768, 0.4, 2, 4), (32768, 0.6, 2, 4),
                                             (100, 0.9, 3, 8), (17, 0.5, 1, 4), (1, 0.4, 2, 4), (0, 0.4, 2, 4)])
def test_span_layout_by_coverage(L, cov, kmin, kmax):
    st, ln = W.span_layout(W.rng(11), L, coverage=cov, kmin=kmin, kmax=kmax)
    _check_spans(st, ln, L, kmin, kmax)
    covered = int(ln.sum())
    # drawn until the target is reached, stopping early only when the next span cannot fit
    assert covered >= int(round(cov * L)) or covered + kmax > L
    assert covered < int(round(cov * L)) + kmax


def test_span_layout_exact_count_and_uniform_gaps():
    st, ln = W.span_layout(W.rng(1), 512, n_spans=40, kmin=2, kmax=4)
    _check_spans(st, ln, 512, 2, 4)
    assert len(st) == 40
    # stars and bars: over many draws every gap (before, between, after) has the same mean
    gaps = []
    for seed in range(400):
        s, k = W.span_layout(W.rng(seed), 64, n_spans=4, kmin=2, kmax=2)
        ends = np.concatenate([[0], s + k])
        nxt = np.concatenate([s, [64]])
        gaps.append(nxt - ends)
    g = np.asarray(gaps, float).mean(axis=0)
    assert np.allclose(g, g.mean(), rtol=0.15)
    with pytest.raises(ValueError):
        W.span_layout(W.rng(0), 5, n_spans=3, kmin=2, kmax=2)


def test_decode_case_structure():
    lens = [1, 15, 16, 17, 300, 0, 4096]
    c = W.decode_case(5, lens=lens, n_q_heads=32, n_kv_heads=8, head_dim=128, n_layers=2, coverage=0.3,
                      spare_pages=3)
    bt = c.block_table.numpy()
    pages = [(L + 15) // 16 for L in lens]
    used = np.concatenate([bt[b, :pages[b]] for b in range(len(lens))])
    assert np.all(bt[bt >= 0] < c.n_pages) and len(np.unique(used)) == len(used) == sum(pages)
    for b in range(len(lens)):
        assert np.all(bt[b, pages[b]:] == -1)
    assert c.n_pages == sum(pages) + 3
    offs, st, ln = c.span_offsets.numpy(), c.span_start.numpy(), c.span_len.numpy()
    assert offs[0] == 0 and offs[-1] == len(st) and np.all(np.diff(offs) >= 0)
    for b, L in enumerate(lens):
        _check_spans(st[offs[b]:offs[b + 1]], ln[offs[b]:offs[b + 1]], L, 2, 4)
    S = len(st)
    assert tuple(c.surrogate_k.shape) == (S, 2, 8, 128) and c.surrogate_k.dtype == torch.bfloat16
    assert tuple(c.pool.shape) == (2, c.n_pages, 2, 8, 16, 128) and tuple(c.q.shape) == (7, 32, 128)
    # physical order differs from logical order
    assert not np.array_equal(used, np.sort(used))


def test_suffix_only_spans_end_at_the_length():
    c = W.decode_case(9, lens=[50, 3, 1, 200], n_q_heads=8, n_kv_heads=2, head_dim=64, coverage=1.0,
                      suffix_only=True)
    offs, st, ln = c.span_offsets.numpy(), c.span_start.numpy(), c.span_len.numpy()
    for b, L in enumerate([50, 3, 1, 200]):
        assert offs[b + 1] - offs[b] == 1
        assert st[offs[b]] + ln[offs[b]] == L


def test_bf16_draws_are_seeded_and_scaled():
    a = W.bf16_normal((1 << 16,), 0.02, 123)
    b = W.bf16_normal((1 << 16,), 0.02, 123)
    c = W.bf16_normal((1 << 16,), 0.02, 124)
    assert torch.equal(a, b) and not torch.equal(a, c)
    assert a.dtype == torch.bfloat16 and abs(a.float().std().item() - 0.02) < 0.001
    u = W.bf16_uniform((1 << 14,), -0.1, 0.1, 5).float()
    lim = torch.tensor(0.1).to(torch.bfloat16).item()    # the bounds rounded to bf16
    assert u.min().item() >= -lim and u.max().item() <= lim
    bits = W.bits(torch.tensor([1.0, -2.0], dtype=torch.bfloat16))
    assert bits.tolist() == [0x3F80, 0xC000]


def test_serving_lengths_follow_the_clipped_lognormal():
    x = W.serving_lengths(W.rng(3), 20000)
    assert x.min() >= 256 and x.max() <= 8192
    assert abs(np.median(x) - 1024) < 40
    # P(X < 256) = Phi(ln(1/4)) ~ 8.3 %, P(X > 8192) = 1 - Phi(ln 8) ~ 1.9 %
    assert abs(np.mean(x == 256) - 0.083) < 0.01 and abs(np.mean(x == 8192) - 0.019) < 0.006


def test_page_allocator_is_first_in_first_out():
    a = W.PageAllocator([7, 3, 9])
    got = a.take([16, 5, 0, 32])
    assert got.tolist() == [7, -1, 3, 9]
    a.give_back([4, 1])
    assert a.take([48, 48]).tolist() == [4, 1]
    with pytest.raises(IndexError):
        a.take([0])


def test_serving_loop_layout_and_free_list():
    sl = W.serving_loop(W.SEEDS["serving"], B=64, n_layers=2, n_q_heads=8, n_kv_heads=2, head_dim=64, steps=40)
    bt = sl.block_table
    used = bt[bt >= 0]
    assert len(np.unique(used)) == len(used)
    assert sorted(used.tolist() + sl.free_pages) == list(range(sl.n_pages))
    for b in range(sl.B):
        assert (bt[b] >= 0).sum() == (int(sl.lens[b]) + 15) // 16
        assert bt.shape[1] * 16 >= int(sl.lens[b]) + 40
    # the rollback draws are reproducible and hit about p of the sequences
    assert sl.rollbacks(5) == sl.rollbacks(5)
    hits = sum(len(sl.rollbacks(s)) for s in range(200))
    assert abs(hits / (200 * 64) - 0.1) < 0.01
    assert all(2 <= k <= 4 for s in range(20) for _, k in sl.rollbacks(s))


def test_random_rules_are_distinct_with_the_requested_counts():
    rules = W.random_rules(17, (300, 200, 100), 50)
    n = (rules >= 0).sum(axis=1)
    assert [int((n == k).sum()) for k in (2, 3, 4)] == [300, 200, 100]
    assert np.all(rules[rules >= 0] < 50)
    for k in (2, 3, 4):
        sub = rules[n == k][:, :k]
        assert len(np.unique(sub, axis=0)) == len(sub)
        assert np.all(rules[n == k][:, k:] == -1)
    assert len(W.rule_tuples(rules)) == len(rules)


def test_rule_prompts_plant_rules_over_about_the_coverage():
    rules = W.random_rules(4, (50, 50, 50), 100000)
    ids = W.rule_prompts(5, rules, B=4, L=2048, vocab=100000, coverage=0.4, lens=[2048, 1000, 2048, 7])
    assert ids.shape == (4, 2048) and np.all(ids[1, 1000:] == -1) and np.all(ids[3, 7:] == -1)
    # with a vocabulary this large, chance rule occurrences are rare: count planted 2..4-grams
    table = set(W.rule_tuples(rules))
    row = ids[0].tolist()
    covered, t = 0, 0
    while t < 2048:
        for k in (4, 3, 2):
            if tuple(row[t:t + k]) in table:
                covered += k
                t += k
                break
        else:
            t += 1
    assert abs(covered / 2048 - 0.4) < 0.01


def test_distill_case_rows_and_stride():
    c = W.distill_case(3, lens=[512, 0, 77], vocab=1001, coverage=0.4)
    assert c.teacher_logits.shape == (589, 1008) and c.teacher_logits.dtype == torch.bfloat16
    offs = c.span_offsets.numpy()
    for b, L in enumerate([512, 0, 77]):
        _check_spans(c.span_start.numpy()[offs[b]:offs[b + 1]], c.span_len.numpy()[offs[b]:offs[b + 1]], L, 2, 4)
