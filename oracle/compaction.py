"""Compressed prompt construction, oracle (test infrastructure only).

App. E ("Prompt Merging") and App. C.5: every selected span is replaced by its
surrogate embedding and the other tokens keep their own static embedding, in
order; the compressed prompt has length L~_p = L_p - sum_{(i,j)} (j - i - 1)
and contiguous positions 0 .. L~_p - 1 (App. J.4, "Compressed-position
convention": [x1, x2, x3, x4] -> [x1, x23, x4] at positions [0, 1, 2]).

Readings: the surrogate (float32, as the merge step returns it) is stored in
the bf16 embedding sequence rounded to nearest, ties to even; prompts are
packed back to back and cu_seqlens holds the prefix sums of the compressed
lengths (the usual variable-length prefill layout).
"""
import numpy as np

from . import bf16
from .spans import check_spans


def build_compressed(table_bits, token_ids, span_offsets, span_start, span_len, surrogates):
    """table_bits [V][d] uint16; token_ids [B][L]; span_offsets [B+1];
    span_start/span_len [S] (positions inside their prompt); surrogates
    [S][d] float32.  Returns (embeds [sum L'][d] uint16, position_ids, cu_seqlens)."""
    token_ids = np.asarray(token_ids)
    B, L = token_ids.shape
    span_offsets = np.asarray(span_offsets)
    span_start = np.asarray(span_start)
    span_len = np.asarray(span_len)
    sur_bits = bf16.from_f32(np.asarray(surrogates, dtype=np.float32))
    rows = []            # per output row: ("tok", id) or ("span", index)
    pos = []
    cu = [0]
    for b in range(B):
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        check_spans(L, span_start[lo:hi], span_len[lo:hi])
        t, i, n = 0, lo, 0
        while t < L:
            if i < hi and t == int(span_start[i]):
                rows.append(("span", i))
                t += int(span_len[i])
                i += 1
            else:
                rows.append(("tok", int(token_ids[b, t])))
                t += 1
            pos.append(n)
            n += 1
        cu.append(cu[-1] + n)
    d = table_bits.shape[1]
    out = np.empty((len(rows), d), dtype=np.uint16)
    for r, (kind, v) in enumerate(rows):
        out[r] = sur_bits[v] if kind == "span" else table_bits[v]
    return out, np.asarray(pos, np.int32), np.asarray(cu, np.int32)
