"""Decode-step KV append of the oracle (test infrastructure only).

App. E ("Decoding-Time Merging and KV-Cache Update") and Fig. 2, step (2):
when no merge rule matches the suffix, the newly generated token is forwarded
through the backbone and its KV state is appended to the cache, one entry per
layer.  For a paged cache that means, per sequence b with L = seq_lens[b]:

  1. entry L lives in page block_table[b][L // P], slot L % P; when L % P == 0
     that page does not exist yet and the caller's allocator supplies it
     (new_pages[b] is written into block_table[b][L // P]);
  2. in every layer, the K and V rows of that slot receive new_k[b][layer] and
     new_v[b][layer];
  3. seq_lens[b] becomes L + 1.

A sequence whose append is impossible (no room in its block-table row, no
page supplied at a page boundary, a page id outside the pool) is left
unchanged and reported; the others are appended.  KV values are raw bf16 bit
patterns, so the result is exact.
"""
import numpy as np


def kv_append(pool, block_table, seq_lens, new_k, new_v, new_pages=None, page_size=16):
    """pool      [n_layers][n_pages][2][Hkv][P][D] uint16 (bf16 bits)
    block_table [B][max_pages] int32
    seq_lens    [B] int32
    new_k/new_v [B][n_layers][Hkv][D] uint16
    new_pages   [B] int32 or None: the page opened by a sequence whose length
                is a multiple of P
    Returns (pool', block_table', seq_lens', rejected) with rejected the
    sorted list of sequences left unchanged."""
    P = page_size
    pool = np.array(pool, copy=True)
    bt = np.array(block_table, dtype=np.int32, copy=True)
    lens = np.array(seq_lens, dtype=np.int32, copy=True)
    n_pages = pool.shape[1]
    rejected = []
    for b in range(bt.shape[0]):
        L = int(lens[b])
        if L < 0 or L >= bt.shape[1] * P:
            rejected.append(b)
            continue
        if L % P == 0:
            page = -1 if new_pages is None else int(new_pages[b])
        else:
            page = int(bt[b, L // P])
        if page < 0 or page >= n_pages:
            rejected.append(b)
            continue
        bt[b, L // P] = page                                  # step 1
        pool[:, page, 0, :, L % P, :] = new_k[b]              # step 2
        pool[:, page, 1, :, L % P, :] = new_v[b]
        lens[b] = L + 1                                       # step 3
    return pool, bt, lens, rejected
