"""The decode loop of a serving engine on the GPU against the oracle.

Every step appends one KV entry per sequence and layer (umim_kv_append),
then each sequence with probability p merges its last k stored entries, the
new one included, into one surrogate entry (umim_kv_rollback of a suffix
span, App. E), then decode attention runs for every layer
(umim_decode_attention).  Each loop also runs with the append and the merge
fused into one umim_decode_append_merge call.

* Small loops: the oracle replays the same steps on a host copy of the cache
  and everything is compared after every step: block tables, lengths, freed
  pages and every valid KV byte bit-exactly, attention outputs within the
  float tolerance.
* The full serving workload (128 sequences with lognormal lengths, 32 layers
  of 32/8 heads, head_dim 128, 256 steps, p = 0.1): the oracle replays the
  steps on a cache whose entries are ids (where each entry came from) instead
  of KV values, which moves exactly as KV bytes do.  Block tables, lengths and
  freed pages are compared after every step; at steps 0, 1, 2, 127 and 255
  the ids are turned back into KV values from the seeded generators, and KV
  bytes and attention outputs are compared for sampled sequences in all
  layers and for all sequences in the first and last layer.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import dev, float_close, umim

pytestmark = pytest.mark.gpu
P = 16


def _spans(rolls, lens, B):
    """CSR suffix spans (start = L - k, k) for the rolled sequences."""
    offs = np.zeros(B + 1, np.int32)
    st, ln = [], []
    ks = dict(rolls)
    for b in range(B):
        offs[b + 1] = offs[b]
        if b in ks:
            k = min(ks[b], int(lens[b]))
            st.append(int(lens[b]) - k)
            ln.append(k)
            offs[b + 1] += 1
    return offs, np.array(st, np.int32), np.array(ln, np.int32)


class GpuLoop:
    """The CUDA path: the library's three calls on device buffers, or with
    fused=True the append and the suffix merge in one umim_decode_append_merge
    call (the released pages then come back one per sequence)."""

    def __init__(self, sl, dv, fused=False):
        self.m = umim()
        self.sl, self.dv, self.fused = sl, dv, fused
        self.pool = sl.init_pool(dv)
        self.bt = torch.from_numpy(sl.block_table.copy()).to(dv)
        self.lens = torch.from_numpy(sl.lens.copy()).to(dv)
        self.status = self.m.new_status(dv)
        kv = self.m.paged_kv(self.pool)
        B, max_pages = sl.block_table.shape
        self.rb_ws = self.m.workspace(self.m.umim_kv_rollback_workspace_size(
            B, B, max_pages, kv.n_layers, kv.n_kv_heads, kv.head_dim), dv)
        self.at_ws = self.m.workspace(self.m.umim_decode_attention_workspace_size(
            B, sl.n_q_heads, sl.n_kv_heads, sl.head_dim), dv)
        self.freed = torch.empty(B * max_pages, dtype=torch.int32, device=dv)
        self.released = torch.empty(B, dtype=torch.int32, device=dv)

    def step(self, step, new_pages, offs, st, ln):
        m, sl, dv = self.m, self.sl, self.dv
        nk, nv = sl.new_entries(step, dv)
        if self.fused:
            B = len(offs) - 1
            merge_k = np.zeros(B, np.int32)
            merge_row = np.full(B, -1, np.int32)
            for b in range(B):
                if offs[b + 1] > offs[b]:
                    merge_k[b], merge_row[b] = ln[offs[b]], offs[b]
            sk, sv = sl.surrogates(step, len(st), dv)
            t = lambda x: torch.from_numpy(x).to(dv)
            m.umim_decode_append_merge(self.pool, self.bt, self.lens, nk, nv, t(new_pages), t(merge_k), t(merge_row),
                                       sk, sv, released=self.released, dev_status=self.status)
            return self._attend(step)
        m.umim_kv_append(self.pool, self.bt, self.lens, nk, nv, torch.from_numpy(new_pages).to(dv),
                         dev_status=self.status)
        sk, sv = sl.surrogates(step, len(st), dv)
        m.umim_kv_rollback(self.pool, self.bt, self.lens, torch.from_numpy(offs).to(dv),
                           torch.from_numpy(st).to(dv), torch.from_numpy(ln).to(dv), sk, sv,
                           freed_pages=self.freed, workspace_buf=self.rb_ws, dev_status=self.status)
        return self._attend(step)

    def _attend(self, step):
        m, sl, dv = self.m, self.sl, self.dv
        outs = []
        for layer in range(sl.n_layers):
            outs.append(m.umim_decode_attention(sl.q(step, layer, dv), self.pool, layer, self.bt, self.lens,
                                                workspace_buf=self.at_ws, dev_status=self.status))
        return outs


def _check_indices(g, o_bt, o_lens, o_freed, step):
    torch.cuda.synchronize()
    assert int(g.status.item()) == 0, f"step {step}: device status {int(g.status.item())}"
    np.testing.assert_array_equal(g.bt.cpu().numpy(), o_bt, err_msg=f"step {step}")
    np.testing.assert_array_equal(g.lens.cpu().numpy(), o_lens, err_msg=f"step {step}")
    if g.fused:
        r = g.released.cpu().numpy()
        assert r[r >= 0].tolist() == list(o_freed), f"step {step}"
        return
    f = g.freed.cpu().numpy()
    assert f[:len(o_freed)].tolist() == list(o_freed), f"step {step}"
    if len(o_freed) < len(f):
        assert f[len(o_freed)] == -1


@pytest.mark.parametrize("fused", [False, True], ids=["three_calls", "fused"])
@pytest.mark.parametrize("seed,B,layers,hq,hkv,d,steps,p", [
    (31, 6, 3, 16, 4, 128, 40, 0.3),
    (32, 5, 2, 8, 2, 64, 36, 0.5),
])
def test_small_serving_loop_matches_oracle_every_step(seed, B, layers, hq, hkv, d, steps, p, fused):
    lens = W.rng(seed).integers(1, 200, size=B).astype(np.int32)
    lens[0] = 16
    sl = W.serving_loop(seed, B=B, n_layers=layers, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, steps=steps, p=p,
                        lens=lens)
    dv = dev()
    g = GpuLoop(sl, dv, fused)
    # every tensor is drawn on the GPU's generator and copied to the host for the oracle
    o_pool = W.bits(sl.init_pool(dv))
    o_bt, o_lens = sl.block_table.copy(), sl.lens.copy()
    alloc = W.PageAllocator(sl.free_pages)
    n_rolled = 0
    for step in range(steps):
        new_pages = alloc.take(o_lens)
        nk, nv = sl.new_entries(step, dv)
        o_pool, o_bt, o_lens, rej = oracle.kv_append(o_pool, o_bt, o_lens, W.bits(nk), W.bits(nv), new_pages)
        assert rej == []
        offs, st, ln = _spans(sl.rollbacks(step), o_lens, B)
        sk, sv = sl.surrogates(step, len(st), dv)
        o_pool, o_bt, o_lens, o_freed = oracle.kv_rollback(o_pool, o_bt, o_lens, offs, st, ln, W.bits(sk),
                                                           W.bits(sv))
        alloc.give_back(o_freed)
        n_rolled += len(st)
        outs = g.step(step, new_pages, offs, st, ln)
        _check_indices(g, o_bt, o_lens, o_freed, step)
        gp = W.bits(g.pool)
        for b in range(B):
            t = np.arange(int(o_lens[b]))
            pg, sl_ = o_bt[b, t // P], t % P
            np.testing.assert_array_equal(gp[:, pg, :, :, sl_, :], o_pool[:, pg, :, :, sl_, :],
                                          err_msg=f"step {step} seq {b}")
        for layer in range(layers):
            want = oracle.decode_attention(W.bits(sl.q(step, layer, dv)), o_pool, layer, o_bt, o_lens)
            float_close(outs[layer].cpu().double().numpy(), want, f"step {step} layer {layer}")
    assert n_rolled > 0


# ---------------------------------------------------------------------------
# the full serving workload, through an id-valued oracle cache
# ---------------------------------------------------------------------------
INIT, APPENDED, SURROGATE = 0, 1, 2
CHECK_STEPS = (0, 1, 2, 127, 255)


def _ids(kind, a, b, n):
    """n entries' ids as [n][1 layer][2][1 head][4] uint16 (K and V rows alike)."""
    e = np.zeros((n, 1, 2, 1, 4), np.uint16)
    e[:, :, :, :, 0] = kind
    e[:, :, :, :, 1] = a
    e[:, :, :, :, 2] = np.asarray(b, np.uint16).reshape(n, 1, 1, 1) if np.ndim(b) else b
    return e


def _id_pool(sl):
    """Initial cache of ids: page p slot s holds (INIT, p, s)."""
    pool = np.zeros((1, sl.n_pages, 2, 1, P, 4), np.uint16)
    pool[..., 0] = INIT
    pool[..., 1] = np.arange(sl.n_pages, dtype=np.uint16).reshape(1, -1, 1, 1, 1)
    pool[..., 2] = np.arange(P, dtype=np.uint16).reshape(1, 1, 1, 1, P)
    return pool


def _materialise(ids, layer, dv, init_layer, draw):
    """KV values [L][2][Hkv][D] (uint16 bits) of a list of ids [L][4], drawn
    again from the seeded generators (draw(kind, step) -> (K, V) bits)."""
    L = ids.shape[0]
    out = np.empty((L,) + tuple(init_layer.shape[1:3]) + (init_layer.shape[4],), np.uint16)
    kind = ids[:, 0]
    sel = np.nonzero(kind == INIT)[0]
    if len(sel):
        pages = torch.from_numpy(ids[sel, 1].astype(np.int64)).to(dv)
        slots = torch.from_numpy(ids[sel, 2].astype(np.int64)).to(dv)
        out[sel] = W.bits(init_layer[pages, :, :, slots, :])            # [n][2][Hkv][D]
    for k in (APPENDED, SURROGATE):
        sel = np.nonzero(kind == k)[0]
        for step in np.unique(ids[sel, 1]):
            kk, vv = draw(k, int(step))
            s2 = sel[ids[sel, 1] == step]
            idx = ids[s2, 2].astype(np.int64)
            out[s2, 0] = kk[idx, layer]
            out[s2, 1] = vv[idx, layer]
    return out


@pytest.mark.parametrize("fused", [False, True], ids=["three_calls", "fused"])
def test_full_serving_workload_matches_oracle(fused):
    sl = W.serving_loop(W.SEEDS["serving"], B=128, n_layers=32, n_q_heads=32, n_kv_heads=8, head_dim=128,
                        steps=256, p=0.1)
    dv = dev()
    g = GpuLoop(sl, dv, fused)
    B = sl.B
    o_pool = _id_pool(sl)
    o_bt, o_lens = sl.block_table.copy(), sl.lens.copy()
    alloc = W.PageAllocator(sl.free_pages)
    cache, n_spans = {}, {}

    def draw(kind, step):
        if (kind, step) not in cache:
            t = sl.new_entries(step, dv) if kind == APPENDED else sl.surrogates(step, n_spans[step], dv)
            cache[(kind, step)] = tuple(W.bits(x) for x in t)
        return cache[(kind, step)]

    sampled = sorted(set([int(np.argmax(sl.lens)), int(np.argmin(sl.lens))] +
                         [int(x) for x in W.rng(99).choice(B, 4, replace=False)]))
    n_rolled = 0
    for step in range(sl.steps):
        new_pages = alloc.take(o_lens)
        aid = _ids(APPENDED, step, np.arange(B), B)
        o_pool, o_bt, o_lens, rej = oracle.kv_append(o_pool, o_bt, o_lens, aid[:, :, 0], aid[:, :, 1], new_pages)
        assert rej == []
        offs, st, ln = _spans(sl.rollbacks(step), o_lens, B)
        S = len(st)
        n_spans[step] = S
        sid = _ids(SURROGATE, step, np.arange(S), S)
        o_pool, o_bt, o_lens, o_freed = oracle.kv_rollback(o_pool, o_bt, o_lens, offs, st, ln, sid[:, :, 0],
                                                           sid[:, :, 1])
        alloc.give_back(o_freed)
        n_rolled += S
        outs = g.step(step, new_pages, offs, st, ln)
        _check_indices(g, o_bt, o_lens, o_freed, step)
        if step not in CHECK_STEPS:
            continue
        for layer in range(sl.n_layers):
            init_layer = sl.init_layer(layer, dv)
            seqs = range(B) if layer in (0, sl.n_layers - 1) else sampled
            q = W.bits(sl.q(step, layer, dv))
            got_out = outs[layer].cpu().double().numpy()
            g_layer = g.pool[layer]
            for b in seqs:
                L = int(o_lens[b])
                t = np.arange(L)
                pg, slot = o_bt[b, t // P], t % P
                ids = o_pool[0, pg, 0, 0, slot, :]                           # [L][4]
                want_kv = _materialise(ids, layer, dv, init_layer, draw)      # [L][2][Hkv][D]
                got_kv = W.bits(g_layer[torch.from_numpy(pg.astype(np.int64)).to(dv), :, :,
                                        torch.from_numpy(slot.astype(np.int64)).to(dv), :])
                np.testing.assert_array_equal(got_kv, want_kv, err_msg=f"step {step} layer {layer} seq {b}")
                # attention of this sequence over the expected cache, laid out contiguously
                n_pg = (L + P - 1) // P
                pool_b = np.zeros((1, n_pg, 2, sl.n_kv_heads, P, sl.head_dim), np.uint16)
                pool_b[0, t // P, :, :, t % P, :] = want_kv
                want = oracle.decode_attention(q[b:b + 1], pool_b, 0, np.arange(n_pg, dtype=np.int32)[None],
                                               np.array([L], np.int32))
                float_close(got_out[b:b + 1], want, f"step {step} layer {layer} seq {b}")
            del init_layer
    assert n_rolled > 0


def test_captured_step_replays_the_eager_fused_loop_bit_for_bit():
    """The fused serving step (update + attention for every layer) captured
    once as a CUDA graph and replayed with each step's inputs copied into its
    static buffers gives, bit for bit, what the eager calls give."""
    B, layers, hq, hkv, d, steps = 6, 3, 16, 4, 128, 30
    lens = W.rng(35).integers(1, 200, size=B).astype(np.int32)
    sl = W.serving_loop(35, B=B, n_layers=layers, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, steps=steps, p=0.5,
                        lens=lens)
    dv = dev()
    m = umim()
    # host bookkeeping of the loop: pages handed out, merges per step
    alloc = W.PageAllocator(sl.free_pages)
    o_lens, o_bt = sl.lens.copy(), sl.block_table.copy()
    o_pool = np.zeros((1, sl.n_pages, 2, 1, 16, 1), np.uint16)   # indices only: values are irrelevant here
    sched = []
    for step in range(steps):
        new_pages = alloc.take(o_lens)
        zeros = np.zeros((B, 1, 1, 1), np.uint16)
        o_pool, o_bt, o_lens, _ = oracle.kv_append(o_pool, o_bt, o_lens, zeros, zeros, new_pages)
        offs, st, ln = _spans(sl.rollbacks(step), o_lens, B)
        S = len(st)
        o_pool, o_bt, o_lens, freed = oracle.kv_rollback(o_pool, o_bt, o_lens, offs, st, ln,
                                                        np.zeros((S, 1, 1, 1), np.uint16),
                                                        np.zeros((S, 1, 1, 1), np.uint16))
        alloc.give_back(freed)
        mk, mr = np.zeros(B, np.int32), np.full(B, -1, np.int32)
        for b in range(B):
            if offs[b + 1] > offs[b]:
                mk[b], mr[b] = ln[offs[b]], offs[b]
        sched.append((new_pages, mk, mr, S))
    t = lambda a: torch.from_numpy(a).to(dv)
    entries = [sl.new_entries(s, dv) for s in range(steps)]
    surs = [sl.surrogates(s, sched[s][3], dv) for s in range(steps)]
    qs = [sl.q(0, layer, dv) for layer in range(layers)]
    ws_a = m.workspace(m.umim_decode_attention_workspace_size(B, hq, hkv, d), dv)

    def fresh():
        return sl.init_pool(dv), t(sl.block_table.copy()), t(sl.lens.copy())

    # eager
    pool, bt, ln_ = fresh()
    status = m.new_status(dv)
    rel = torch.empty(B, dtype=torch.int32, device=dv)
    eager = []
    for s in range(steps):
        np_, mk, mr, S = sched[s]
        m.umim_decode_append_merge(pool, bt, ln_, entries[s][0], entries[s][1], t(np_), t(mk), t(mr), surs[s][0],
                                   surs[s][1], released=rel, dev_status=status)
        outs = [m.umim_decode_attention(qs[l], pool, l, bt, ln_, workspace_buf=ws_a, dev_status=status)
                for l in range(layers)]
        eager.append(([o.clone() for o in outs], rel.clone()))
    e_pool, e_bt, e_len = pool.clone(), bt.clone(), ln_.clone()
    # captured once, replayed every step
    pool, bt, ln_ = fresh()
    n_max = max(1, max(x[3] for x in sched))
    st_nk, st_nv = torch.empty_like(entries[0][0]), torch.empty_like(entries[0][1])
    st_np, st_mk, st_mr = (torch.empty(B, dtype=torch.int32, device=dv) for _ in range(3))
    st_sk = torch.zeros((n_max, layers, hkv, d), dtype=torch.bfloat16, device=dv)
    st_sv = torch.zeros_like(st_sk)
    g_outs = [torch.empty_like(qs[0]) for _ in range(layers)]
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        m.umim_decode_append_merge(pool, bt, ln_, st_nk, st_nv, st_np, st_mk, st_mr, st_sk, st_sv, released=rel,
                                   dev_status=status)
        for l in range(layers):
            m.umim_decode_attention(qs[l], pool, l, bt, ln_, out=g_outs[l], workspace_buf=ws_a, dev_status=status)
    for s in range(steps):
        np_, mk, mr, S = sched[s]
        st_nk.copy_(entries[s][0])
        st_nv.copy_(entries[s][1])
        st_np.copy_(t(np_))
        st_mk.copy_(t(mk))
        st_mr.copy_(t(mr))
        if S:
            st_sk[:S].copy_(surs[s][0])
            st_sv[:S].copy_(surs[s][1])
        graph.replay()
        for l in range(layers):
            assert torch.equal(g_outs[l], eager[s][0][l]), (s, l)
        assert torch.equal(rel, eager[s][1]), s
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert torch.equal(bt, e_bt) and torch.equal(ln_, e_len)
    tl = e_len.cpu().numpy()
    btn = e_bt.cpu().numpy()
    gp, ep = W.bits(pool), W.bits(e_pool)
    for b in range(B):
        tt = np.arange(int(tl[b]))
        pg, slot = btn[b, tt // 16], tt % 16
        np.testing.assert_array_equal(gp[:, pg, :, :, slot, :], ep[:, pg, :, :, slot, :])
