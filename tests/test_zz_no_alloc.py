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

