"""The per-layer decode step on the GPU against the oracle.

A decode step calls umim_decode_layer_step once per layer, in layer order,
each call writing that layer's new (or surrogate) entry and returning that
layer's attention over the updated cache; the last call commits the block
tables and lengths.  The oracle's reading of one step: kv_append of the new
entries, then kv_rollback of each merging sequence's suffix span (App. E,
"Decoding-Time Merging and KV-Cache Update"), then decode_attention per layer
over the resulting cache.  Block tables, lengths, released pages and every
valid KV byte are compared bit for bit after every step; attention outputs
within the float tolerance, every layer of every step.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, float_close, oracle_append_merge, umim

pytestmark = pytest.mark.gpu


def _free_pages(bt, n_pages):
    used = set(int(x) for x in bt[bt >= 0].ravel())
    return [p for p in range(n_pages) if p not in used]


def _run_steps(seed, lens, hq, hkv, d, layers, steps, p_merge=0.35, permute_rows=False, extra_rows=0):
    m = umim()
    dv = dev()
    B = len(lens)
    extra = (steps + 15) // 16 + 1
    c = W.decode_case(seed, lens=lens, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, n_layers=layers, coverage=0.0,
                      spare_pages=B * extra, extra_max_pages=extra)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    o_pool, o_bt, o_lens = W.bits(c.pool), c.block_table.numpy(), c.seq_lens.numpy()
    alloc = W.PageAllocator(_free_pages(o_bt, c.n_pages))
    r = W.rng(seed + 7)
    status = m.new_status(dv)
    ws = m.workspace(m.umim_decode_layer_step_workspace_size(B, hkv, d), dv)
    released = torch.empty(B, dtype=torch.int32, device=dv)
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dv)
    n_merged = 0
    for step in range(steps):
        nk = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 4 * step, dv)
        nv = W.bf16_normal((B, layers, hkv, d), 1.0, seed * 1000 + 4 * step + 1, dv)
        q = W.bf16_normal((layers, B, hq, d), 1.0, seed * 1000 + 4 * step + 2, dv)
        new_pages = alloc.take(o_lens)
        merge_k = np.where(r.random(B) < p_merge, r.integers(1, 17, size=B), 0).astype(np.int32)
        merge_k = np.minimum(merge_k, o_lens + 1).astype(np.int32)
        S = int((merge_k > 0).sum())
        R = max(S + extra_rows, 1)
        rows = r.permutation(R)[:S] if permute_rows else np.arange(S)
        merge_row = np.full(B, -1, np.int32)
        merge_row[merge_k > 0] = rows
        sk = W.bf16_normal((R, layers, hkv, d), 1.0, seed * 1000 + 500 + 2 * step, dv)
        sv = W.bf16_normal((R, layers, hkv, d), 1.0, seed * 1000 + 501 + 2 * step, dv)
        outs = []
        for layer in range(layers):
            outs.append(m.umim_decode_layer_step(
                q[layer], pool, layer, bt, sl, nk[:, layer], nv[:, layer], t(new_pages), t(merge_k), t(merge_row),
                sk[:, layer].contiguous(), sv[:, layer].contiguous(), commit=layer == layers - 1,
                released=released, workspace_buf=ws, dev_status=status))
        # the oracle's step: append, suffix rollback (surrogates in sequence order), attention per layer
        order = rows.astype(np.int64)
        o_pool, o_bt, o_lens, o_rel = oracle_append_merge(o_pool, o_bt, o_lens, W.bits(nk), W.bits(nv), new_pages,
                                                           merge_k, W.bits(sk)[order], W.bits(sv)[order])
        alloc.give_back([p for p in o_rel if p >= 0])
        n_merged += S
        torch.cuda.synchronize()
        assert int(status.item()) == 0, f"step {step}"
        np.testing.assert_array_equal(bt.cpu().numpy(), o_bt, err_msg=f"step {step}")
        np.testing.assert_array_equal(sl.cpu().numpy(), o_lens, err_msg=f"step {step}")
        np.testing.assert_array_equal(released.cpu().numpy(), o_rel, err_msg=f"step {step}")
        gp = W.bits(pool)
        for b in range(B):
            tt = np.arange(int(o_lens[b]))
            pg, slot = o_bt[b, tt // 16], tt % 16
            np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], o_pool[:, pg, :, :, slot, :],
                                          err_msg=f"step {step} seq {b}")
        qb = W.bits(q)
        for layer in range(layers):
            want = oracle.decode_attention(qb[layer], o_pool, layer, o_bt, o_lens)
            float_close(outs[layer].cpu().double().numpy(), want, f"step {step} layer {layer}")
    assert n_merged > 0


@pytest.mark.parametrize("seed,lens,hq,hkv,d,layers,steps", [
    # page phases: empty, 1, 15, 16, 17, 31, 32 entries, ...
    (51, [0, 1, 15, 16, 17, 31, 32, 100, 255, 256], 32, 8, 128, 3, 12),
    (52, [3, 16, 47, 64, 2047], 8, 2, 64, 2, 10),
    # few long sequences with G = 7: every segment split over many warps (merged by the last to finish)
    (53, [4000, 5, 33, 1200], 28, 4, 128, 2, 6),
    # one KV head per query head (G = 1) and G = 16
    (54, [40, 16, 0, 700], 8, 8, 64, 2, 6),
    (55, [90, 300, 16], 32, 2, 128, 2, 6),
])
def test_layer_steps_match_append_rollback_attention(seed, lens, hq, hkv, d, layers, steps):
    _run_steps(seed, lens, hq, hkv, d, layers, steps)


def test_surrogate_rows_in_any_order():
    """merge_row may point anywhere in a larger surrogate array."""
    _run_steps(56, [20, 47, 16, 300, 2, 64], 16, 4, 128, 2, 8, p_merge=0.6, permute_rows=True, extra_rows=5)


def test_many_sequences_one_layer():
    """A batch of 300 sequences of every page phase (more sequences than SMs)."""
    _run_steps(57, list(range(0, 1200, 4)), 8, 2, 64, 1, 3)


def test_rejected_sequences_are_left_unchanged():
    """Sequences whose step cannot happen are neither written nor committed
    (UMIM_ERR_INVALID_ARG), their output is attention over the unchanged
    cache; the other sequences take their step."""
    m = umim()
    dv = dev()
    lens = [10, 20, 3, 40, 32, 16]
    Hq, Hkv, D, NL = 8, 4, 128, 2
    c = W.decode_case(58, lens=lens, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, n_layers=NL, coverage=0.0,
                      spare_pages=4, extra_max_pages=1)
    B = len(lens)
    pool, bt, sl = c.pool.to(dv), c.block_table.to(dv), c.seq_lens.to(dv)
    free = _free_pages(c.block_table.numpy(), c.n_pages)
    nk = W.bf16_normal((B, NL, Hkv, D), 1.0, 911, dv)
    nv = W.bf16_normal((B, NL, Hkv, D), 1.0, 912, dv)
    q = W.bf16_normal((NL, B, Hq, D), 1.0, 913, dv)
    sk = W.bf16_normal((2, NL, Hkv, D), 1.0, 914, dv)
    sv = W.bf16_normal((2, NL, Hkv, D), 1.0, 915, dv)
    # 0: k = 17; 1: row outside the surrogates; 2: k > L + 1; 3: a good merge (row 1);
    # 4: a page boundary without a page; 5: a page boundary with a good page
    merge_k = torch.tensor([17, 2, 5, 3, 0, 0], dtype=torch.int32, device=dv)
    merge_row = torch.tensor([0, 2, 0, 1, -1, -1], dtype=torch.int32, device=dv)
    new_pages = torch.tensor([-1, -1, -1, -1, -1, free[0]], dtype=torch.int32, device=dv)
    status = m.new_status(dv)
    released = torch.empty(B, dtype=torch.int32, device=dv)
    ws = m.workspace(m.umim_decode_layer_step_workspace_size(B, Hkv, D), dv)
    outs = [m.umim_decode_layer_step(q[l], pool, l, bt, sl, nk[:, l], nv[:, l], new_pages, merge_k, merge_row,
                                     sk[:, l].contiguous(), sv[:, l].contiguous(), commit=l == NL - 1,
                                     released=released, workspace_buf=ws, dev_status=status) for l in range(NL)]
    torch.cuda.synchronize()
    assert int(status.item()) == 1   # UMIM_ERR_INVALID_ARG
    assert sl.cpu().tolist() == [10, 20, 3, 40 + 1 - 3 + 1, 32, 17]
    obt = c.block_table.numpy()
    np.testing.assert_array_equal(bt.cpu().numpy()[[0, 1, 2, 4]], obt[[0, 1, 2, 4]])
    assert bt.cpu().numpy()[5, 1] == free[0]
    assert released.cpu().tolist() == [-1, -1, -1, -1, -1, -1]
    gp, op = W.bits(pool), W.bits(c.pool)
    for b in (0, 1, 2, 4):
        tt = np.arange(lens[b])
        pg, slot = obt[b, tt // 16], tt % 16
        np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], op[:, pg, :, :, slot, :])
    p38 = obt[3, 38 // 16]
    np.testing.assert_array_equal(gp[:, p38, 0, :, 38 % 16, :], W.bits(sk)[1])
    np.testing.assert_array_equal(gp[:, p38, 1, :, 38 % 16, :], W.bits(sv)[1])
    # outputs: the rejected sequences see their unchanged caches, the others their step
    got_bt, got_lens = bt.cpu().numpy(), sl.cpu().numpy()
    qb = W.bits(q)
    for l in range(NL):
        want = oracle.decode_attention(qb[l], gp, l, got_bt, got_lens)
        float_close(outs[l].cpu().double().numpy(), want, f"layer {l}")


def test_equals_the_three_call_step_on_the_serving_shape():
    """Two steps of the serving loop's shape (128 sequences of lognormal
    length, 32 layers of 32/8 heads) through the per-layer call and through
    umim_decode_append_merge + umim_decode_attention: identical caches,
    tables and lengths; attention outputs within the tolerance of each other,
    and the first and last layers against the oracle."""
    m = umim()
    dv = dev()
    sl_ = W.serving_loop(W.SEEDS["serving"], B=128, n_layers=32, n_q_heads=32, n_kv_heads=8, head_dim=128,
                         steps=2, p=0.3)
    B, NL = sl_.B, sl_.n_layers
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dv)
    pools = [sl_.init_pool(dv) for _ in range(2)]
    bts = [t(sl_.block_table) for _ in range(2)]
    lens = [t(sl_.lens) for _ in range(2)]
    alloc = W.PageAllocator(sl_.free_pages)
    status = m.new_status(dv)
    ws = m.workspace(m.umim_decode_layer_step_workspace_size(B, 8, 128), dv)
    ws_a = m.workspace(m.umim_decode_attention_workspace_size(B, 32, 8, 128), dv)
    rel = [torch.empty(B, dtype=torch.int32, device=dv) for _ in range(2)]
    h_lens = sl_.lens.copy()
    for step in range(2):
        nk, nv = sl_.new_entries(step, dv)
        new_pages = alloc.take(h_lens)
        rolls = dict(sl_.rollbacks(step))
        merge_k = np.array([min(rolls.get(b, 0), int(h_lens[b]) + 1) for b in range(B)], np.int32)
        S = int((merge_k > 0).sum())
        merge_row = np.where(merge_k > 0, np.cumsum(merge_k > 0) - 1, -1).astype(np.int32)
        sk, sv = sl_.surrogates(step, max(S, 1), dv)
        qs = [sl_.q(step, layer, dv) for layer in range(NL)]
        a_out = []
        for layer in range(NL):
            a_out.append(m.umim_decode_layer_step(qs[layer], pools[0], layer, bts[0], lens[0], nk[:, layer],
                                                  nv[:, layer], t(new_pages), t(merge_k), t(merge_row),
                                                  sk[:, layer].contiguous(), sv[:, layer].contiguous(),
                                                  commit=layer == NL - 1, released=rel[0], workspace_buf=ws,
                                                  dev_status=status))
        m.umim_decode_append_merge(pools[1], bts[1], lens[1], nk, nv, t(new_pages), t(merge_k), t(merge_row), sk,
                                   sv, released=rel[1], dev_status=status)
        b_out = [m.umim_decode_attention(qs[layer], pools[1], layer, bts[1], lens[1], workspace_buf=ws_a,
                                         dev_status=status) for layer in range(NL)]
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        np.testing.assert_array_equal(bts[0].cpu().numpy(), bts[1].cpu().numpy())
        np.testing.assert_array_equal(lens[0].cpu().numpy(), lens[1].cpu().numpy())
        np.testing.assert_array_equal(rel[0].cpu().numpy(), rel[1].cpu().numpy())
        alloc.give_back([p for p in rel[0].cpu().tolist() if p >= 0])
        h_lens = lens[0].cpu().numpy()
        o_bt = bts[0].cpu().numpy()
        # both paths write the same slots of the same pages: the whole pools agree bit for bit
        # (compared on the device; the 33 GB pools stay there)
        assert torch.equal(pools[0].view(torch.int16), pools[1].view(torch.int16)), f"step {step}: pools differ"
        for layer in range(NL):
            float_close(a_out[layer].cpu().double().numpy(), b_out[layer].cpu().double().numpy(),
                        f"step {step} layer {layer} against the three-call step")
        for layer in (0, NL - 1):
            g_layer = W.bits(pools[0][layer:layer + 1])
            want = oracle.decode_attention(W.bits(qs[layer]), g_layer, 0, o_bt, h_lens)
            float_close(a_out[layer].cpu().double().numpy(), want, f"step {step} layer {layer} against the oracle")
