"""Decode attention through the allocation-free entry point.

Callers such as a serving engine that has already handed all GPU memory to
its own allocator, or a plug-in that may not allocate outside its host
framework's arena, cannot supply a workspace.  umim_decode_attention_static
serves them from a scratch array built into the library.  This checks,
through the C ABI, that it returns what the workspace-based
umim_decode_attention returns, on two calls in a row (the second call finds
the first call's leftovers in the shared array), and that a batch too large
for the array is refused before anything runs.
"""
import pytest
import torch

import workloads as W
from helpers import case_to_dev, dev, float_close, umim

pytestmark = pytest.mark.gpu


def test_static_scratch_matches_workspace_entry_point_twice():
    m = umim()
    d = dev()
    cases = [
        W.decode_case(301, lens=[1000, 17, 0, 4096, 333, 64], n_q_heads=32, n_kv_heads=8, head_dim=128,
                      n_layers=2, n_spans=[0] * 6),
        W.decode_case(302, lens=[511, 2, 2048], n_q_heads=28, n_kv_heads=4, head_dim=64, n_layers=1,
                      n_spans=[0] * 3),
    ]
    for c in cases:
        g = case_to_dev(c, d)
        for layer in range(c.n_layers):
            status = m.new_status(d)
            want = m.umim_decode_attention(g["q"], g["pool"], layer, g["bt"], g["lens"], dev_status=status)
            got1 = m.umim_decode_attention_static(g["q"], g["pool"], layer, g["bt"], g["lens"], dev_status=status)
            got2 = m.umim_decode_attention_static(g["q"], g["pool"], layer, g["bt"], g["lens"], dev_status=status)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            float_close(got1.cpu().double().numpy(), want.cpu().double().numpy(), "first call")
            float_close(got2.cpu().double().numpy(), want.cpu().double().numpy(), "second call")


def test_batch_too_large_for_the_scratch_array_is_refused():
    m = umim()
    d = dev()
    # 65536 sequences x 16 KV heads need far more partial-result space than the array holds
    B, Hq, Hkv, D = 65536, 16, 16, 128
    pool = torch.zeros((1, 1, 2, Hkv, 16, D), dtype=torch.bfloat16, device=d)
    q = torch.zeros((B, Hq, D), dtype=torch.bfloat16, device=d)
    bt = torch.zeros((B, 1), dtype=torch.int32, device=d)
    lens = torch.ones(B, dtype=torch.int32, device=d)
    with pytest.raises(m.UmimError) as e:
        m.umim_decode_attention_static(q, pool, 0, bt, lens)
    assert e.value.code == 5   # UMIM_ERR_WORKSPACE



def _largest_batch_that_fits(m, Hq, Hkv, D):
    """The largest batch whose scratch, sized like the workspace of
    umim_decode_attention on this device, fits in the library's array."""
    lo, hi = 1, 1
    while m.umim_decode_attention_workspace_size(hi, Hq, Hkv, D) <= m.STATIC_SCRATCH_BYTES:
        lo, hi = hi, 2 * hi
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if m.umim_decode_attention_workspace_size(mid, Hq, Hkv, D) <= m.STATIC_SCRATCH_BYTES:
            lo = mid
        else:
            hi = mid
    return lo


def test_batch_just_under_the_array_limit_matches_the_oracle():
    """A batch whose plan and partials nearly fill the array (computed from the
    workspace size at this device's SM count) still runs and matches the
    oracle; one more sequence is refused."""
    import numpy as np
    import oracle
    m = umim()
    d = dev()
    Hq, Hkv, D = 32, 8, 128
    B = _largest_batch_that_fits(m, Hq, Hkv, D)
    assert m.umim_decode_attention_workspace_size(B + 1, Hq, Hkv, D) > m.STATIC_SCRATCH_BYTES
    lens = W.rng(303).integers(0, 70, size=B).tolist()
    c = W.decode_case(303, lens=lens, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=D, n_spans=[0] * B)
    g = case_to_dev(c, d)
    status = m.new_status(d)
    got = m.umim_decode_attention_static(g["q"], g["pool"], 0, g["bt"], g["lens"], dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    want = oracle.decode_attention(W.bits(c.q), W.bits(c.pool), 0, c.block_table.numpy(), c.seq_lens.numpy())
    float_close(got.cpu().double().numpy(), want, "batch at the array limit")
    q1 = torch.zeros((B + 1, Hq, D), dtype=torch.bfloat16, device=d)
    bt1 = torch.zeros((B + 1, g["bt"].shape[1]), dtype=torch.int32, device=d)
    l1 = torch.zeros(B + 1, dtype=torch.int32, device=d)
    with pytest.raises(m.UmimError) as e:
        m.umim_decode_attention_static(q1, g["pool"], 0, bt1, l1)
    assert e.value.code == 5   # UMIM_ERR_WORKSPACE


def test_warm_calls_reserve_no_device_memory_and_keep_the_current_device():
    """After the first call on the device (the set-up), further calls leave the
    device's free memory unchanged, and the caller's current device is the
    same after each call."""
    m = umim()
    d = dev()
    c = W.decode_case(304, lens=[300, 5, 1200], n_q_heads=16, n_kv_heads=4, head_dim=64, n_spans=[0] * 3)
    g = case_to_dev(c, d)
    out = torch.empty_like(g["q"])
    status = m.new_status(d)
    m.umim_decode_attention_static(g["q"], g["pool"], 0, g["bt"], g["lens"], out=out, dev_status=status)
    torch.cuda.synchronize()
    before_dev = torch.cuda.current_device()
    free0 = torch.cuda.mem_get_info(d)[0]
    for _ in range(3):
        m.umim_decode_attention_static(g["q"], g["pool"], 0, g["bt"], g["lens"], out=out, dev_status=status)
        assert torch.cuda.current_device() == before_dev
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info(d)[0] == free0
    assert int(status.item()) == 0
