"""Decode attention on the GPU against the oracle, within max-abs 1e-2 and
relative L2 2e-3 (bf16 in, fp32 accumulate, bf16 out)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from helpers import case_to_dev, dev, float_close, oracle_rollback, umim

pytestmark = pytest.mark.gpu


def _attend(c, layer=0, scale=0.0, pool=None, bt=None, lens=None):
    m = umim()
    d = dev()
    g = case_to_dev(c, d)
    if pool is not None:
        g["pool"], g["bt"], g["lens"] = pool, bt, lens
    status = m.new_status(d)
    out = m.umim_decode_attention(g["q"], g["pool"], layer, g["bt"], g["lens"], scale=scale, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return out.cpu()


CASES = [
    # seed, lens, Hq, Hkv, D, layers
    (1, [432], 8, 2, 64, 1),                                # tiny shape after rollback
    (2, [1, 2, 15, 16, 17, 31, 33, 1000, 0], 32, 8, 128, 2),
    (3, [5000, 3], 28, 4, 128, 1),                          # G = 7
    (4, [700, 1200, 64], 16, 16, 128, 3),                   # G = 1
    (5, [300, 2500], 16, 1, 64, 1),                         # G = 16
    (6, [4097, 16 * 300], 8, 4, 64, 2),
]


@pytest.mark.parametrize("seed,lens,hq,hkv,d,layers", CASES)
def test_attention_matches_oracle(seed, lens, hq, hkv, d, layers):
    c = W.decode_case(seed, lens=lens, n_q_heads=hq, n_kv_heads=hkv, head_dim=d, n_layers=layers,
                      n_spans=[0] * len(lens), spare_pages=3)
    for layer in range(layers):
        out = _attend(c, layer)
        ref = oracle.decode_attention(W.bits(c.q), W.bits(c.pool), layer, c.block_table.numpy(),
                                      c.seq_lens.numpy())
        float_close(out.double().numpy(), ref, f"layer {layer}")


def test_explicit_scale():
    c = W.decode_case(7, lens=[500, 77], n_q_heads=8, n_kv_heads=2, head_dim=128, n_spans=[0, 0])
    out = _attend(c, 0, scale=0.25)
    ref = oracle.decode_attention(W.bits(c.q), W.bits(c.pool), 0, c.block_table.numpy(), c.seq_lens.numpy(),
                                  scale=0.25)
    float_close(out.double().numpy(), ref)


def test_empty_sequences_give_zero():
    c = W.decode_case(8, lens=[0, 40, 0], n_q_heads=8, n_kv_heads=2, head_dim=64, n_spans=[0, 0, 0])
    out = _attend(c).float()
    assert torch.all(out[0] == 0) and torch.all(out[2] == 0)


def test_garbage_past_the_end_is_ignored():
    """Slots after the last entry may hold anything, NaN included."""
    c = W.decode_case(9, lens=[21, 5], n_q_heads=4, n_kv_heads=1, head_dim=128, n_spans=[0, 0])
    pool = c.pool.clone()
    bt = c.block_table.numpy()
    pool[0, bt[0, 1], :, :, 5:, :] = float("nan")
    pool[0, bt[1, 0], :, :, 5:, :] = float("inf")
    c.pool = pool
    out = _attend(c)
    assert torch.isfinite(out.float()).all()
    ref = oracle.decode_attention(W.bits(c.q), W.bits(pool), 0, bt, c.seq_lens.numpy())
    float_close(out.double().numpy(), ref)


def test_after_gpu_rollback():
    """Rollback then attention, both on the GPU, against the oracle's rollback
    followed by the oracle's attention."""
    m = umim()
    d = dev()
    c = W.decode_case(10, lens=[1000, 333, 4096], n_q_heads=32, n_kv_heads=8, head_dim=128, n_layers=2,
                      coverage=0.35)
    g = case_to_dev(c, d)
    status = m.new_status(d)
    m.umim_kv_rollback(g["pool"], g["bt"], g["lens"], g["offs"], g["st"], g["ln"], g["sk"], g["sv"],
                       dev_status=status)
    out = m.umim_decode_attention(g["q"], g["pool"], 1, g["bt"], g["lens"], dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    rp, rbt, rl, _ = oracle_rollback(c)
    ref = oracle.decode_attention(W.bits(c.q), rp, 1, rbt, rl)
    float_close(out.cpu().double().numpy(), ref)


@pytest.mark.parametrize("name", ["llama8b_layer", "long_context", "long_context_tr40"])
def test_full_size_configs_after_rollback(name):
    seed = W.SEEDS[name]
    if name == "llama8b_layer":
        c = W.decode_case(seed, lens=[4096] * 16, n_q_heads=32, n_kv_heads=8, head_dim=128, coverage=0.3)
    elif name == "long_context":
        c = W.decode_case(seed, lens=[32768] * 4, n_q_heads=28, n_kv_heads=4, head_dim=128, coverage=0.4)
    else:
        c = W.decode_case(seed, lens=[32768] * 4, n_q_heads=28, n_kv_heads=4, head_dim=128, coverage=0.6)
    rp, rbt, rl, _ = oracle_rollback(c)
    d = dev()
    pool = torch.from_numpy(rp.view(np.int16)).view(torch.bfloat16).to(d)
    out = _attend(c, 0, pool=pool, bt=torch.from_numpy(rbt).to(d), lens=torch.from_numpy(rl).to(d))
    ref = oracle.decode_attention(W.bits(c.q), rp, 0, rbt, rl)
    float_close(out.double().numpy(), ref, name)


def test_serving_shape_sampled_layers():
    """32-layer pool, lognormal lengths (median 1024, clipped 256..8192), one
    suffix rollback per sequence with probability 0.1: a few layers checked."""
    r = W.rng(W.SEEDS["serving"])
    lens = W.serving_lengths(r, 12)
    c = W.decode_case(W.SEEDS["serving"], lens=lens, n_q_heads=32, n_kv_heads=8, head_dim=128, n_layers=32,
                      coverage=0.1, suffix_only=True)
    m = umim()
    d = dev()
    g = case_to_dev(c, d)
    status = m.new_status(d)
    m.umim_kv_rollback(g["pool"], g["bt"], g["lens"], g["offs"], g["st"], g["ln"], g["sk"], g["sv"],
                       dev_status=status)
    outs = {}
    for layer in (0, 13, 31):
        outs[layer] = m.umim_decode_attention(g["q"], g["pool"], layer, g["bt"], g["lens"], dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    rp, rbt, rl, _ = oracle_rollback(c)
    np.testing.assert_array_equal(g["lens"].cpu().numpy(), rl)
    for layer, out in outs.items():
        ref = oracle.decode_attention(W.bits(c.q), rp, layer, rbt, rl)
        float_close(out.cpu().double().numpy(), ref, f"layer {layer}")


def test_calls_leave_the_callers_current_device_unchanged():
    """Every call makes its stream's device current only while it runs: the
    caller's current device is the same afterwards (on a side stream too)."""
    m = umim()
    d = dev()
    c = W.decode_case(71, lens=[100, 37], n_q_heads=8, n_kv_heads=2, head_dim=64, n_spans=[0, 0])
    g = case_to_dev(c, d)
    before = torch.cuda.current_device()
    side = torch.cuda.Stream(d)
    status = m.new_status(d)
    with torch.cuda.stream(side):
        m.umim_decode_attention(g["q"], g["pool"], 0, g["bt"], g["lens"], dev_status=status, stream=side)
    assert torch.cuda.current_device() == before
    m.umim_decode_attention(g["q"], g["pool"], 0, g["bt"], g["lens"], dev_status=status)
    assert torch.cuda.current_device() == before
    torch.cuda.synchronize()
    assert int(status.item()) == 0
