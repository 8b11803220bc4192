"""Merge-rule matching and the surrogate lookup of the oracle (test
infrastructure only).

App. E ("Rule Matching"): rules are token n-grams, n in {4, 3, 2}.

Prompt merging scans the token ids from left to right.  At a position the
candidate n-grams starting there are tried longest first (4, then 3, then
2); the first one that is a rule becomes a span and the scan continues at
the first token after it; when none is a rule the scan moves on by one
token.  The spans are therefore non-overlapping and in order.

Decoding-time merging applies the same longest-first test, after each newly
generated token, to the raw-token suffix that ends at that token.  The state
kept for a sequence is its generated tokens, where a merged span counts as
one opaque marker: a later suffix never reaches across a marker, so merges
never overlap or nest.  Generation starts with an empty state (the prompt is
not part of it).  A merge of n tokens replaces the n - 1 cached entries of
the suffix plus the new token by one surrogate entry: the cache update's k
(stored entries replaced once the new token's entry is in) is n.

The lookup: a surrogate depends only on the tokens of its span, so one
surrogate per rule can be computed ahead of time and fetched by rule id
(App. E, potential engineering optimizations); fetching is indexing.

Rules are given as a list of n-grams; rule id = position in that list.  The
matcher reads them through a dict from n-gram to rule id.
"""
import numpy as np

LENGTHS = (4, 3, 2)   # longest first


def rule_dict(rules):
    """rules: sequence of token tuples (length 2..4), distinct.
    Returns {tuple: rule id}."""
    d = {}
    for r, g in enumerate(rules):
        g = g if type(g) is tuple else tuple(int(x) for x in g)
        if not 2 <= len(g) <= 4:
            raise ValueError(f"rule {r} has length {len(g)}")
        if g in d:
            raise ValueError(f"rule {r} repeats rule {d[g]}")
        d[g] = r
    return d


def match_prompt(tokens, rules):
    """Left-to-right, longest-first matching of one prompt.
    tokens: sequence of token ids; rules: {tuple: rule id}.
    Returns a list of (start, n, rule id), in order."""
    tokens = [int(x) for x in tokens]
    spans = []
    i = 0
    while i < len(tokens):
        for n in LENGTHS:
            g = tuple(tokens[i:i + n])
            if len(g) == n and g in rules:
                spans.append((i, n, rules[g]))
                i += n
                break
        else:
            i += 1
    return spans


def match_prompts(token_ids, lens, rules):
    """A batch of prompts [B][L] with lengths lens[b] (tokens past the length
    are ignored) -> (span_offsets [B+1], span_start [S], span_len [S],
    span_rule [S]) as int32 arrays, starts relative to their prompt."""
    offs, st, ln, rl = [0], [], [], []
    for b in range(len(lens)):
        for (s, n, r) in match_prompt(token_ids[b][:int(lens[b])], rules):
            st.append(s)
            ln.append(n)
            rl.append(r)
        offs.append(len(st))
    i32 = lambda x: np.asarray(x, dtype=np.int32)
    return i32(offs), i32(st), i32(ln), i32(rl)


class SuffixState:
    """One sequence's decoding state: the raw generated tokens since the
    start of generation or the last merge (only the last three matter, since
    a rule has at most four tokens and the fourth is the new one)."""

    def __init__(self, raw=()):
        self.raw = [int(x) for x in raw][-3:]

    def step(self, y, rules):
        """Feed the newly generated token y.  Returns (n, rule id) of the
        merge it completes, or (0, -1)."""
        cand = self.raw + [int(y)]
        for n in LENGTHS:
            if n <= len(cand):
                g = tuple(cand[-n:])
                if g in rules:
                    self.raw = []            # the merged span is now one marker
                    return n, rules[g]
        self.raw = cand[-3:]
        return 0, -1


def match_suffixes(states, new_tokens, rules):
    """One decode step for a batch: per sequence (merge_k, rule id), plus for
    the merging sequences their rank in sequence order (merge_row, -1 when
    none) and the rule ids in that order."""
    B = len(states)
    merge_k = np.zeros(B, np.int32)
    merge_rule = np.full(B, -1, np.int32)
    merge_row = np.full(B, -1, np.int32)
    rows_rule = []
    for b in range(B):
        n, r = states[b].step(new_tokens[b], rules)
        if n:
            merge_k[b], merge_rule[b] = n, r
            merge_row[b] = len(rows_rule)
            rows_rule.append(r)
    return merge_k, merge_rule, merge_row, np.asarray(rows_rule, np.int32)


def lookup(lut, rule_ids):
    """Surrogate rows by rule id: lut [R][d] -> [n][d]."""
    return np.asarray(lut)[np.asarray(rule_ids, dtype=np.int64)]
