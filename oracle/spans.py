"""Span bookkeeping of the oracle (test infrastructure only).

A span (s, k) of a sequence of length L covers positions s .. s+k-1 and is
replaced by one unit.  Following App. J.4 ("Structural effect under RoPE"),
r(t) is the number of positions removed before position t, and a position
that survives moves to pi(t) = t - r(t).  A span's single replacement unit
takes the compressed index of its first position (App. C.5 example:
[x1, x2, x3, x4] -> [e(x1), z23, e(x4)] at positions [0, 1, 2]).
"""
import numpy as np


def check_spans(L: int, starts, lens):
    """Spans must be sorted, non-overlapping, k >= 1 and inside [0, L)."""
    prev_end = 0
    for s, k in zip(starts, lens):
        s, k = int(s), int(k)
        if k < 1 or s < prev_end or s + k > L:
            raise ValueError(f"invalid span ({s},{k}) for length {L}")
        prev_end = s + k


def compressed_length(L: int, lens) -> int:
    """L' = L - sum over spans of (k - 1)  (App. E, "Prompt Merging")."""
    return int(L) - int(sum(int(k) - 1 for k in lens))


def span_metadata(L: int, starts, lens):
    """For each position t < L: its compressed index, or the index of the unit
    that replaces it.  Returns (new_index[L], is_span_start[L], is_covered[L])."""
    check_spans(L, starts, lens)
    new_index = np.empty(L, dtype=np.int64)
    covered = np.zeros(L, dtype=bool)
    first = np.zeros(L, dtype=bool)
    removed = 0
    t = 0
    i = 0
    starts = [int(s) for s in starts]
    lens = [int(k) for k in lens]
    while t < L:
        if i < len(starts) and t == starts[i]:
            k = lens[i]
            for u in range(t, t + k):
                new_index[u] = t - removed
                covered[u] = True
            first[t] = True
            removed += k - 1
            t += k
            i += 1
        else:
            new_index[t] = t - removed
            t += 1
    return new_index, first, covered
