"""Pins of the oracle's rule matching and surrogate lookup (App. E "Rule
Matching", "Prompt Merging", "Decoding-Time Merging and KV-Cache Update").

The matchers are pinned against things other than themselves:
  * a hand-worked example (tests/golden/rule_matching_example.json);
  * an independent checker of the conditions that define the greedy prompt
    scan (in-order, non-overlapping rule spans; at every position the scan
    stops at, no longer rule starts there and, where it advances by one, no
    rule starts at all) -- these conditions have exactly one solution;
  * closed forms (every 2-gram a rule; every 2- and 3-gram a rule);
  * for rule sets of 2-grams only, decoding-time merging over a token stream
    equals prompt matching over the same stream;
  * the decode state against a list model with merged markers;
  * the cache-length rule L_C' = L_C - (n - 1) + 1;
  * the lookup against running the (separately pinned) merge module on the
    matched spans: surrogates depend only on a span's tokens.
"""
import json
import os

import numpy as np
import pytest

from oracle import rules as R
from oracle.merge import merge_spans

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "rule_matching_example.json")


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def check_greedy(tokens, rules, spans):
    """True when spans is the left-to-right longest-first scan of tokens;
    written from the defining conditions, not by rescanning."""
    L = len(tokens)
    starts = {s: (n, r) for (s, n, r) in spans}
    prev_end = 0
    for (s, n, r) in spans:
        if s < prev_end or not 2 <= n <= 4 or s + n > L:
            return False
        if rules.get(tuple(tokens[s:s + n])) != r:
            return False
        prev_end = s + n

    def longest_at(p):
        best = 0
        for n in (2, 3, 4):
            if p + n <= L and tuple(tokens[p:p + n]) in rules:
                best = n
        return best

    p = 0
    while p < L:
        if p in starts:
            n = starts.pop(p)[0]
            if longest_at(p) != n:
                return False
            p += n
        else:
            if longest_at(p) != 0:
                return False
            p += 1
    return not starts   # every span start was a position the scan stops at


def test_golden_prompt_example():
    g = _golden()
    rules = R.rule_dict(g["rules"])
    spans = R.match_prompt(g["prompt"]["tokens"], rules)
    assert [list(x) for x in spans] == g["prompt"]["spans"]
    L = len(g["prompt"]["tokens"])
    assert L - sum(n - 1 for (_, n, _) in spans) == g["prompt"]["compressed_length"]


def test_golden_decode_example():
    g = _golden()
    rules = R.rule_dict(g["rules"])
    st = R.SuffixState()
    C = g["decode"]["cache_length_before"]
    for t, y in enumerate(g["decode"]["tokens"]):
        n, r = st.step(y, rules)
        assert n == g["decode"]["merge_n"][t] and r == g["decode"]["merge_rule"][t], t
        C = C + 1 if n == 0 else C - (n - 1) + 1
        assert C == g["decode"]["cache_length_after"][t]


def _random_rules(rng, alphabet, n_rules):
    out = set()
    while len(out) < n_rules:
        n = int(rng.integers(2, 5))
        out.add(tuple(int(x) for x in rng.integers(0, alphabet, size=n)))
    return sorted(out)


@pytest.mark.parametrize("seed", range(6))
def test_prompt_scan_satisfies_the_greedy_conditions(seed):
    rng = np.random.default_rng(seed)
    alphabet = [3, 4, 6, 10, 20, 50][seed]
    rules = R.rule_dict(_random_rules(rng, alphabet, min(40, alphabet ** 2)))
    for _ in range(60):
        toks = [int(x) for x in rng.integers(0, alphabet, size=int(rng.integers(0, 120)))]
        spans = R.match_prompt(toks, rules)
        assert check_greedy(toks, rules, spans)


def test_checker_rejects_plausible_mistakes():
    """The checker is strict enough to catch the usual slips of a scan."""
    rules = R.rule_dict([(1, 2), (1, 2, 3), (2, 3)])
    toks = [1, 2, 3, 2, 3]
    good = R.match_prompt(toks, rules)
    assert good == [(0, 3, 1), (3, 2, 2)] and check_greedy(toks, rules, good)
    assert not check_greedy(toks, rules, [(0, 2, 0), (3, 2, 2)])            # shortest first
    assert not check_greedy(toks, rules, [(0, 3, 1), (1, 2, 2), (3, 2, 2)])  # advance by one after a match
    assert not check_greedy(toks, rules, [(0, 3, 1)])                       # stopped early
    assert not check_greedy(toks, rules, [(0, 3, 0), (3, 2, 2)])            # wrong rule id


@pytest.mark.parametrize("L", [0, 1, 2, 3, 7, 64, 65])
def test_every_pair_a_rule_gives_consecutive_pairs(L):
    rules = R.rule_dict([(a, b) for a in range(2) for b in range(2)])
    toks = [int(x) for x in np.random.default_rng(L).integers(0, 2, size=L)]
    spans = R.match_prompt(toks, rules)
    assert [(s, n) for (s, n, _) in spans] == [(2 * i, 2) for i in range(L // 2)]


@pytest.mark.parametrize("L", [2, 3, 4, 5, 9, 10, 11])
def test_every_pair_and_triple_a_rule_gives_triples_then_the_rest(L):
    rules = R.rule_dict([(a, b) for a in range(2) for b in range(2)] +
                        [(a, b, c) for a in range(2) for b in range(2) for c in range(2)])
    toks = [0] * L
    spans = R.match_prompt(toks, rules)
    want = [(3 * i, 3) for i in range(L // 3)] + ([(3 * (L // 3), 2)] if L % 3 == 2 else [])
    assert [(s, n) for (s, n, _) in spans] == want


def test_no_rules_or_short_prompts_give_no_spans():
    assert R.match_prompt([1, 2, 3], {}) == []
    rules = R.rule_dict([(1, 2)])
    assert R.match_prompt([], rules) == [] and R.match_prompt([1], rules) == []


@pytest.mark.parametrize("seed", range(4))
def test_decode_with_pair_rules_equals_prompt_matching(seed):
    rng = np.random.default_rng(100 + seed)
    alphabet = 5
    rules = R.rule_dict(sorted({tuple(int(x) for x in rng.integers(0, alphabet, 2)) for _ in range(8)}))
    toks = [int(x) for x in rng.integers(0, alphabet, size=200)]
    st, got = R.SuffixState(), []
    for t, y in enumerate(toks):
        n, r = st.step(y, rules)
        if n:
            got.append((t - n + 1, n, r))
    assert got == R.match_prompt(toks, rules)


@pytest.mark.parametrize("seed", range(4))
def test_decode_state_against_a_list_with_markers(seed):
    """The generated state as the paper keeps it: a list of raw tokens and
    MERGED markers; a suffix qualifies only if it holds no marker."""
    rng = np.random.default_rng(200 + seed)
    alphabet = 4
    rules = R.rule_dict(_random_rules(rng, alphabet, 20))
    MERGED = object()
    state, st = [], R.SuffixState()
    for y in rng.integers(0, alphabet, size=300):
        y = int(y)
        state.append(y)
        want = (0, -1)
        for n in (4, 3, 2):
            tail = state[-n:]
            if len(tail) == n and all(x is not MERGED for x in tail) and tuple(tail) in rules:
                want = (n, rules[tuple(tail)])
                state = state[:-n] + [MERGED]
                break
        assert st.step(y, rules) == want


def test_batch_helpers_agree_with_single_calls():
    rng = np.random.default_rng(7)
    rules = R.rule_dict(_random_rules(rng, 5, 25))
    B, L = 6, 40
    toks = rng.integers(0, 5, size=(B, L))
    lens = np.array([40, 0, 1, 17, 39, 23])
    offs, st, ln, rl = R.match_prompts(toks, lens, rules)
    for b in range(B):
        one = R.match_prompt(toks[b][:lens[b]], rules)
        assert list(zip(st[offs[b]:offs[b + 1]], ln[offs[b]:offs[b + 1]], rl[offs[b]:offs[b + 1]])) == one
    states = [R.SuffixState() for _ in range(B)]
    twins = [R.SuffixState() for _ in range(B)]
    for t in range(30):
        y = rng.integers(0, 5, size=B)
        k, r, row, rows = R.match_suffixes(states, y, rules)
        single = [twins[b].step(y[b], rules) for b in range(B)]
        assert [(int(k[b]), int(r[b])) for b in range(B)] == single
        assert list(rows) == [r[b] for b in range(B) if k[b]]
        assert [int(row[b]) for b in range(B) if k[b]] == list(range(len(rows)))


def test_lookup_of_precomputed_surrogates_equals_merging_the_matched_spans():
    """Surrogates depend only on the span's tokens (App. E): merging every
    rule once and fetching by rule id gives what merging the matched spans
    gives."""
    rng = np.random.default_rng(11)
    V, d, h = 12, 8, 4
    rules_list = _random_rules(rng, V, 15)
    rules = R.rule_dict(rules_list)
    table = rng.integers(0, 1 << 16, size=(V, d), dtype=np.uint16) & 0x3FFF   # finite bf16 bit patterns
    w = dict(w_kv=rng.normal(0, 0.3, (d, d)), b_kv=rng.normal(0, 0.1, d), w_o=rng.normal(0, 0.3, (d, d)),
             b_o=rng.normal(0, 0.1, d), query=rng.normal(0, 1, (h, d // h)),
             ln_kv_gamma=1 + rng.normal(0, 0.05, d), ln_kv_beta=rng.normal(0, 0.05, d),
             ln_o_gamma=1 + rng.normal(0, 0.05, d), ln_o_beta=rng.normal(0, 0.05, d))
    flat = np.concatenate([np.asarray(g) for g in rules_list]).astype(np.int64)
    offs = np.concatenate([[0], np.cumsum([len(g) for g in rules_list])])
    lut = merge_spans(table, flat, offs, w, h)
    toks = [int(x) for x in rng.integers(0, V, size=200)]
    spans = R.match_prompt(toks, rules)
    assert spans
    s_flat = np.concatenate([toks[s:s + n] for (s, n, _) in spans]).astype(np.int64)
    s_offs = np.concatenate([[0], np.cumsum([n for (_, n, _) in spans])])
    direct = merge_spans(table, s_flat, s_offs, w, h)
    np.testing.assert_array_equal(R.lookup(lut, [r for (_, _, r) in spans]), direct)


def test_repeated_or_malformed_rules_are_refused():
    with pytest.raises(ValueError):
        R.rule_dict([(1, 2), (3, 4), (1, 2)])
    with pytest.raises(ValueError):
        R.rule_dict([(1,)])
    with pytest.raises(ValueError):
        R.rule_dict([(1, 2, 3, 4, 5)])
