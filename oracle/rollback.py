"""KV-cache rollback and compaction of the oracle (test infrastructure only).

App. E ("Decoding-Time Merging and KV-Cache Update") and App. C.6: when a span
is merged, the KV entries stored for its tokens are cropped and a single KV
state computed from the surrogate takes their place, so the cache length goes
from L_C to L_C - (n - 1) + 1 (Fig. 2 caption: the span's several KV
entries give way to one merged entry).

This restates that operation for a paged cache and for any number of sorted,
non-overlapping spans per sequence (the paper crops a suffix; spans placed
anywhere are the same replace-k-by-one operation with the tail shifted left):

  1. read the sequence's entries e_0 .. e_{L-1} in logical order
     (entry t lives in page block_table[t // P], slot t % P, in every layer);
  2. build the new list: entries outside spans are kept byte for byte; a span
     (s, k) contributes one entry whose bytes are the given surrogate K/V;
  3. write the new list back into the SAME physical pages in logical order
     (new entry j -> page block_table[j // P], slot j % P);
  4. pages p in [ceil(L'/P), ceil(L/P)) no longer hold entries: their ids are
     reported, in ascending p, sequence after sequence, and block_table[p]
     becomes -1;
  5. seq_len becomes L' = L - sum (k - 1).

Here k counts STORED entries replaced (the paper's n - 1 when the newest token
is not yet cached; n when it is).  Slots of the last page at or beyond L' are
left as they are and are not part of the result.  KV bytes are handled as raw
bf16 bit patterns, so the result is exact.

Position-aware variant (App. J.4, compressed positions pi(t) = t - r(t), and
its RoPE discussion): the cache stores keys already rotated for their
position, so a kept entry that moves from t to pi(t) carries a key rotated
for t.  With rope_inv_freq (the angular frequencies w_m, m < rotary_dim / 2)
every moved kept entry's K rows (all layers and KV heads) are rotated by
-r(t) w_m on the pairs (m, m + rotary_dim / 2) (the half-split pairing of
Llama-style RoPE), which gives the key the rotation of its compressed
position: R(pi(t)) k = R(-r(t)) R(t) k.  Computed in float64 and rounded to
bf16 (ties to even); V rows, columns at or beyond rotary_dim, surrogate
entries and entries that do not move are unchanged.
"""
import numpy as np

from . import bf16
from .spans import check_spans, compressed_length


def rerotate_keys(k_bits, shift, inv_freq, rotary_dim):
    """K rows [..][D] (bf16 bits) rotated by -shift * w_m on the pairs
    (m, m + rotary_dim/2): x' = x cos + y sin, y' = y cos - x sin."""
    k = bf16.to_f64(k_bits)
    half = rotary_dim // 2
    ang = float(shift) * np.asarray(inv_freq, dtype=np.float64)[:half]
    c, s = np.cos(ang), np.sin(ang)
    x, y = k[..., :half], k[..., half:rotary_dim]
    out = np.array(k_bits, copy=True)
    out[..., :half] = bf16.from_f64(x * c + y * s)
    out[..., half:rotary_dim] = bf16.from_f64(y * c - x * s)
    return out


def kv_rollback(pool, block_table, seq_lens, span_offsets, span_start, span_len,
                surrogate_k, surrogate_v, page_size=16, rope_inv_freq=None, rotary_dim=None):
    """pool         [n_layers][n_pages][2][Hkv][P][D] uint16 (bf16 bits)
    block_table  [B][max_pages] int32
    seq_lens     [B] int32
    span_offsets [B+1], span_start [S], span_len [S] int32
    surrogate_k/v [S][n_layers][Hkv][D] uint16
    rope_inv_freq [rotary_dim/2] (float32 values) or None: re-rotate moved keys
    rotary_dim   even, <= D (default D)
    Returns (pool', block_table', seq_lens', freed_pages list)."""
    P = page_size
    pool = np.array(pool, copy=True)
    bt = np.array(block_table, dtype=np.int32, copy=True)
    lens = np.array(seq_lens, dtype=np.int32, copy=True)
    span_offsets = np.asarray(span_offsets)
    span_start = np.asarray(span_start)
    span_len = np.asarray(span_len)
    n_layers, n_pages = pool.shape[0], pool.shape[1]
    B = bt.shape[0]
    # validate everything before touching anything
    for b in range(B):
        L = int(lens[b])
        if L < 0 or L > bt.shape[1] * P:
            raise ValueError("seq_len out of range")
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        check_spans(L, span_start[lo:hi], span_len[lo:hi])
        used = bt[b, :(L + P - 1) // P]
        if np.any(used < 0) or np.any(used >= n_pages):
            raise ValueError("block table entry out of range")
    D = pool.shape[5]
    if rope_inv_freq is not None:
        rotary_dim = D if rotary_dim is None else int(rotary_dim)
        if rotary_dim % 2 or not 0 < rotary_dim <= D or len(rope_inv_freq) < rotary_dim // 2:
            raise ValueError("rotary_dim")

    def kept(run, shift):
        """entries of a kept run [n][layers][2][Hkv][D]; moved runs re-rotated."""
        if rope_inv_freq is None or shift == 0 or len(run) == 0:
            return list(run)
        run = np.array(run, copy=True)
        run[:, :, 0] = rerotate_keys(run[:, :, 0], shift, rope_inv_freq, rotary_dim)
        return list(run)

    # [page][slot][layer][K|V][Hkv][D] view of the pool (writes go through it)
    view = pool.transpose(1, 4, 0, 2, 3, 5)
    freed = []
    for b in range(B):
        L = int(lens[b])
        lo, hi = int(span_offsets[b]), int(span_offsets[b + 1])
        if hi == lo:
            continue
        # step 1: logical entries
        t_all = np.arange(L)
        entries = view[bt[b, t_all // P], t_all % P]           # [L][layers][2][Hkv][D]
        # step 2: the new list, left to right: the kept entries before each
        # span, then the span's surrogate entry, then the entries after the
        # last span
        new = []
        t = 0
        r = 0   # positions removed before the current run
        for i in range(lo, hi):
            s, k = int(span_start[i]), int(span_len[i])
            new.extend(kept(entries[t:s], r))
            new.append(np.stack([surrogate_k[i], surrogate_v[i]], axis=1))  # [layers][2][Hkv][D]
            t = s + k
            r += k - 1
        new.extend(kept(entries[t:L], r))
        new = np.stack(new)
        Lp = len(new)
        assert Lp == compressed_length(L, span_len[lo:hi])
        # step 3: write back into the same pages, logical order
        j_all = np.arange(Lp)
        view[bt[b, j_all // P], j_all % P] = new
        # step 4: release pages that no longer hold entries
        for p in range((Lp + P - 1) // P, (L + P - 1) // P):
            freed.append(int(bt[b, p]))
            bt[b, p] = -1
        # step 5
        lens[b] = Lp
    return pool, bt, lens, freed
