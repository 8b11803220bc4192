"""Pins of the oracle's decode-step append (App. E, Fig. 2 step (2)).

The append is pinned against things other than itself:
  * a logical-list model of the cache (a Python list of entries per sequence,
    read back through the block table slot by slot);
  * identities with the rollback oracle (itself pinned by the worked example
    and the length formula): appending x and then replacing that one entry by
    y is appending y; appending n entries and then merging them into one
    surrogate is appending the surrogate, and releases exactly the pages the
    appends opened;
  * the serving step of the decode loop (append, then with some probability
    merge the last k stored entries) against list operations.
"""
import numpy as np
import pytest

import oracle
from oracle.rollback import kv_rollback

P = 16


def _case(seed, lens, n_layers=2, hkv=2, d=8, spare=8, extra_pages=2):
    r = np.random.default_rng(seed)
    B = len(lens)
    pages = [(L + P - 1) // P for L in lens]
    max_pages = max(pages + [1]) + extra_pages
    n_pages = sum(pages) + spare
    perm = r.permutation(n_pages).astype(np.int32)
    bt = np.full((B, max_pages), -1, np.int32)
    k = 0
    for b in range(B):
        for p in range(pages[b]):
            bt[b, p] = perm[k]
            k += 1
    free = [int(x) for x in perm[k:]]
    pool = r.integers(0, 1 << 16, size=(n_layers, n_pages, 2, hkv, P, d), dtype=np.uint16)
    return pool, bt, np.asarray(lens, np.int32), free


def _entry(r, B, n_layers, hkv, d):
    return (r.integers(0, 1 << 16, size=(B, n_layers, hkv, d), dtype=np.uint16),
            r.integers(0, 1 << 16, size=(B, n_layers, hkv, d), dtype=np.uint16))


def _logical(pool, bt, L):
    """Entries of one sequence in logical order, slot by slot: [L][layers][2][Hkv][D]."""
    out = []
    for t in range(L):
        out.append(pool[:, bt[t // P], :, :, t % P, :])
    return np.stack(out) if out else np.zeros((0,) + pool.shape[:1] + pool.shape[2:4] + pool.shape[5:],
                                               pool.dtype)


def _pages_for(lens, free):
    """The allocator: a page for every sequence at a page boundary, in order."""
    new_pages = np.full(len(lens), -1, np.int32)
    for b, L in enumerate(lens):
        if L % P == 0:
            new_pages[b] = free.pop(0)
    return new_pages


def test_append_matches_logical_list_model():
    r = np.random.default_rng(1)
    lens = [0, 1, 15, 16, 17, 31, 32, 47]
    pool, bt, L, free = _case(2, lens, spare=32, extra_pages=4)
    model = [list(_logical(pool, bt[b], lens[b])) for b in range(len(lens))]
    for step in range(40):
        nk, nv = _entry(r, len(lens), pool.shape[0], pool.shape[3], pool.shape[5])
        new_pages = _pages_for([int(x) for x in L], free)
        pool, bt, L, rej = oracle.kv_append(pool, bt, L, nk, nv, new_pages)
        assert rej == []
        for b in range(len(lens)):
            model[b].append(np.stack([nk[b], nv[b]], axis=1))
            got = _logical(pool, bt[b], int(L[b]))
            assert int(L[b]) == lens[b] + step + 1
            assert np.array_equal(got, np.stack(model[b]))


def test_page_opened_only_at_boundary():
    r = np.random.default_rng(3)
    lens = [15, 16, 32, 5]
    pool, bt, L, free = _case(4, lens)
    nk, nv = _entry(r, 4, pool.shape[0], pool.shape[3], pool.shape[5])
    new_pages = np.array([free[0], free[1], free[2], free[3]], np.int32)
    pool2, bt2, L2, rej = oracle.kv_append(pool, bt, L, nk, nv, new_pages)
    assert rej == []
    assert np.array_equal(bt2[0], bt[0]) and np.array_equal(bt2[3], bt[3])   # mid-page: new_pages ignored
    assert bt2[1, 1] == free[1] and bt2[2, 2] == free[2]
    assert np.array_equal(np.delete(bt2[1], 1), np.delete(bt[1], 1))
    # nothing outside the written slots changed
    changed = np.argwhere(pool2 != pool)
    for layer, page, kv, h, slot, col in changed:
        hits = [b for b in range(4) if bt2[b, lens[b] // P] == page and lens[b] % P == slot]
        assert len(hits) == 1


def test_append_then_replace_by_one_entry_is_appending_that_entry():
    r = np.random.default_rng(5)
    lens = [7, 16, 33, 0, 64]
    pool, bt, L, free = _case(6, lens)
    x_k, x_v = _entry(r, 5, pool.shape[0], pool.shape[3], pool.shape[5])
    y_k, y_v = _entry(r, 5, pool.shape[0], pool.shape[3], pool.shape[5])
    new_pages = _pages_for(lens, list(free))
    a_pool, a_bt, a_L, _ = oracle.kv_append(pool, bt, L, x_k, x_v, new_pages)
    offs = np.arange(6, dtype=np.int32)
    a_pool, a_bt, a_L, freed = kv_rollback(a_pool, a_bt, a_L, offs, L.copy(), np.ones(5, np.int32), y_k, y_v)
    b_pool, b_bt, b_L, _ = oracle.kv_append(pool, bt, L, y_k, y_v, new_pages)
    assert freed == []
    assert np.array_equal(a_bt, b_bt) and np.array_equal(a_L, b_L)
    for b in range(5):
        assert np.array_equal(_logical(a_pool, a_bt[b], int(a_L[b])), _logical(b_pool, b_bt[b], int(b_L[b])))


@pytest.mark.parametrize("n", [2, 3, 4, 17])
def test_appending_n_then_merging_them_is_appending_the_surrogate(n):
    r = np.random.default_rng(7 + n)
    lens = [14, 15, 16, 30, 1]
    pool, bt, L, free = _case(8, lens, spare=40, extra_pages=4)
    B = len(lens)
    alloc = list(free)
    opened = [[] for _ in range(B)]
    a_pool, a_bt, a_L = pool, bt, L
    for _ in range(n):
        cur = [int(x) for x in a_L]
        new_pages = _pages_for(cur, alloc)
        for b in range(B):
            if new_pages[b] >= 0:
                opened[b].append((cur[b] // P, int(new_pages[b])))
        nk, nv = _entry(r, B, pool.shape[0], pool.shape[3], pool.shape[5])
        a_pool, a_bt, a_L, _ = oracle.kv_append(a_pool, a_bt, a_L, nk, nv, new_pages)
    s_k, s_v = _entry(r, B, pool.shape[0], pool.shape[3], pool.shape[5])
    offs = np.arange(B + 1, dtype=np.int32)
    a_pool, a_bt, a_L, freed = kv_rollback(a_pool, a_bt, a_L, offs, L.copy(), np.full(B, n, np.int32), s_k, s_v)
    # the same surrogate appended directly, with the allocator's first pages
    direct_pages = _pages_for(lens, list(free))
    b_pool, b_bt, b_L, _ = oracle.kv_append(pool, bt, L, s_k, s_v, direct_pages)
    assert np.array_equal(a_L, b_L)
    for b in range(B):
        assert np.array_equal(_logical(a_pool, a_bt[b], int(a_L[b])), _logical(b_pool, b_bt[b], int(b_L[b])))
    # released: the pages the appends opened beyond the one the surrogate needs, in order
    want = []
    for b in range(B):
        keep = (lens[b] + 1 + P - 1) // P
        want += [page for (p, page) in opened[b] if p >= keep]
    assert freed == want


def test_rejected_sequences_are_left_unchanged():
    r = np.random.default_rng(11)
    lens = [32, 5, 16, 48]       # max_pages = 3: the last row is full
    pool, bt, L, free = _case(12, lens, extra_pages=0)
    assert bt.shape[1] == 3
    nk, nv = _entry(r, 4, pool.shape[0], pool.shape[3], pool.shape[5])
    new_pages = np.array([-1, -1, pool.shape[1], 0], np.int32)   # 0: none given; 2: outside the pool
    pool2, bt2, L2, rej = oracle.kv_append(pool, bt, L, nk, nv, new_pages)
    assert rej == [0, 2, 3]
    assert list(L2) == [32, 6, 16, 48]
    for b in (0, 2, 3):
        assert np.array_equal(bt2[b], bt[b])
        assert np.array_equal(_logical(pool2, bt2[b], lens[b]), _logical(pool, bt[b], lens[b]))


def test_serving_steps_match_list_operations():
    """The decode loop's step (append one entry, then with probability p merge
    the last k stored entries into one surrogate) against a list model."""
    r = np.random.default_rng(13)
    lens = [3, 16, 40, 100]
    B = len(lens)
    pool, bt, L, free = _case(14, lens, spare=64, extra_pages=6)
    alloc = list(free)
    model = [list(_logical(pool, bt[b], lens[b])) for b in range(B)]
    for step in range(60):
        cur = [int(x) for x in L]
        nk, nv = _entry(r, B, pool.shape[0], pool.shape[3], pool.shape[5])
        pool, bt, L, rej = oracle.kv_append(pool, bt, L, nk, nv, _pages_for(cur, alloc))
        assert rej == []
        for b in range(B):
            model[b].append(np.stack([nk[b], nv[b]], axis=1))
        roll = [b for b in range(B) if r.random() < 0.3]
        ks = [int(r.integers(2, 5)) for _ in roll]
        if roll:
            offs = np.zeros(B + 1, np.int32)
            starts, klen = [], []
            for b in range(B):
                offs[b + 1] = offs[b]
                if b in roll:
                    k = min(ks[roll.index(b)], int(L[b]))
                    starts.append(int(L[b]) - k)
                    klen.append(k)
                    offs[b + 1] += 1
            s_k, s_v = _entry(r, len(roll), pool.shape[0], pool.shape[3], pool.shape[5])
            pool, bt, L, freed = kv_rollback(pool, bt, L, offs, np.array(starts, np.int32),
                                             np.array(klen, np.int32), s_k, s_v)
            alloc.extend(freed)
            for j, b in enumerate(roll):
                del model[b][len(model[b]) - klen[j]:]
                model[b].append(np.stack([s_k[j], s_v[j]], axis=1))
        for b in range(B):
            assert int(L[b]) == len(model[b])
            assert np.array_equal(_logical(pool, bt[b], int(L[b])), np.stack(model[b]))
            used = (int(L[b]) + P - 1) // P
            assert np.all(bt[b, used:] == -1) and np.all(bt[b, :used] >= 0)
