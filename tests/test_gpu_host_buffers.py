"""tp_decode_host / tp_prefill_host: the attention calls with host Q, O, LSE.

They run the same kernels as tp_decode_ex / tp_prefill on library staging,
so their results must equal the device-buffer calls' bit for bit (the
device calls are themselves compared with the oracle in test_gpu_parity and
test_gpu_prefill). Consecutive host calls alternate two staging slots with
the copies on streams of their own; the cases below make calls overlap,
reuse one host buffer across calls, mix in device-buffer calls and use
pageable memory.
"""
import numpy as np
import pytest
import torch

import paper_2508_17445_gb300 as tp
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2508_17445_gb300 import build
    build.build()


def _forest(script):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=script.upper_bound_blocks(32) + 64,
                  device=DEV)
    ids = f.replay(script.ops, kv_fn=lambda kv_id: script.kv(kv_id, DEV))
    return f, ids


def _queries(rows, heads, seed, pinned=True):
    g = torch.Generator(device="cpu").manual_seed(seed)
    q = torch.randn(rows, heads.num_q_heads, heads.head_dim, generator=g).to(torch.bfloat16)
    return q.pin_memory() if pinned else q


def _empty_like_host(rows, heads, pinned=True):
    o = torch.empty(rows, heads.num_q_heads, heads.head_dim, dtype=torch.bfloat16)
    lse = torch.empty(rows, heads.num_q_heads, dtype=torch.float32)
    return (o.pin_memory(), lse.pin_memory()) if pinned else (o, lse)


def _device_decode(f, leaves, q_host, flags=0):
    O, LSE = f.decode(leaves, q_host.to(DEV), flags=flags)
    f.sync()
    return O.cpu(), LSE.cpu()


def _same(a, b):
    return a.shape == b.shape and torch.equal(a.view(torch.int16) if a.dtype == torch.bfloat16 else a,
                                              b.view(torch.int16) if b.dtype == torch.bfloat16 else b)


@pytest.mark.parametrize("flags", [0, tp.TP_MMA_SYNC])
def test_consecutive_host_decodes_equal_device_decodes(flags):
    s = workloads.qwen7b(seed=1, n_prompts=2)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    n = len(leaves)
    qs = [_queries(n, s.heads, seed) for seed in range(3)]
    refs = [_device_decode(f, leaves, q, flags) for q in qs]
    outs = [_empty_like_host(n, s.heads) for _ in qs]
    for q, (o, lse) in zip(qs, outs):  # three calls in flight: both staging slots, overlapped copies
        tp.tp_decode_host(f.handle, leaves, q, o, lse, flags)
    f.sync()
    for (o, lse), (o_ref, lse_ref) in zip(outs, refs):
        assert _same(o, o_ref) and _same(lse, lse_ref)
    f.close()


def test_host_buffer_reused_across_calls_holds_the_last_result():
    s = workloads.random_tree(seed=3, heads=workloads.Heads(28, 4, 128), n_prompts=2)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    n = len(leaves)
    qa, qb = _queries(n, s.heads, 10), _queries(n, s.heads, 11)
    ref_b = _device_decode(f, leaves, qb)
    o, lse = _empty_like_host(n, s.heads)
    tp.tp_decode_host(f.handle, leaves, qa, o, lse)
    tp.tp_decode_host(f.handle, leaves, qb, o, lse)
    f.sync()
    assert _same(o, ref_b[0]) and _same(lse, ref_b[1])
    f.close()


def test_host_and_device_calls_interleave():
    s = workloads.wide_prefix(seed=2, n_prompts=1)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    n = len(leaves)
    q1, q2 = _queries(n, s.heads, 20), _queries(n, s.heads, 21)
    ref1, ref2 = _device_decode(f, leaves, q1), _device_decode(f, leaves, q2)
    o1, l1 = _empty_like_host(n, s.heads)
    o2, l2 = _empty_like_host(n, s.heads)
    tp.tp_decode_host(f.handle, leaves, q1, o1, l1)
    O_dev, L_dev = f.decode(leaves, q2.to(DEV))  # a device-buffer call between two host calls
    tp.tp_decode_host(f.handle, leaves, q2, o2, l2)
    f.sync()
    assert _same(o1, ref1[0]) and _same(l1, ref1[1])
    assert _same(o2, ref2[0]) and _same(l2, ref2[1])
    assert _same(O_dev.cpu(), ref2[0])
    f.close()


def test_pageable_host_memory():
    s = workloads.tiny(seed=4)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    n = len(leaves)
    q = _queries(n, s.heads, 30, pinned=False)
    ref = _device_decode(f, leaves, q)
    o, lse = _empty_like_host(n, s.heads, pinned=False)
    tp.tp_decode_host(f.handle, leaves, q, o, lse)
    f.sync()
    assert _same(o, ref[0]) and _same(lse, ref[1])
    f.close()


def test_growing_batches_regrow_the_staging():
    s = workloads.qwen7b(seed=5, n_prompts=2)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    for n in (3, len(leaves), 7, len(leaves)):
        q = _queries(n, s.heads, 40 + n)
        ref = _device_decode(f, leaves[:n], q)
        o, lse = _empty_like_host(n, s.heads)
        tp.tp_decode_host(f.handle, leaves[:n], q, o, lse)
        f.sync()
        assert _same(o, ref[0]) and _same(lse, ref[1])
    f.close()


@pytest.mark.parametrize("flags", [0, tp.TP_MMA_SYNC])
def test_host_prefill_equals_device_prefill(flags):
    s = workloads.segment_prefill(seed=6, n_prompts=2, prompt_len=700, fanout=3, seg_len=300)
    f, ids = _forest(s)
    nodes = [ids[x] for x in s.leaves]
    counts = [300, 1, 0, 150, 299, 300][:len(nodes)]
    total = sum(counts)
    qs = [_queries(total, s.heads, seed) for seed in (50, 51)]
    refs = []
    for q in qs:
        O = torch.empty(q.shape, dtype=torch.bfloat16, device=DEV)
        L = torch.empty(total, s.heads.num_q_heads, dtype=torch.float32, device=DEV)
        tp.tp_prefill(f.handle, nodes, counts, q.to(DEV), O, L, flags)
        f.sync()
        refs.append((O.cpu(), L.cpu()))
    outs = [_empty_like_host(total, s.heads) for _ in qs]
    for q, (o, lse) in zip(qs, outs):
        tp.tp_prefill_host(f.handle, nodes, counts, q, o, lse, flags)
    f.sync()
    for (o, lse), (o_ref, lse_ref) in zip(outs, refs):
        assert _same(o, o_ref) and _same(lse, lse_ref)
    f.close()


def test_forest_wrappers():
    s = workloads.segment_prefill(seed=7, n_prompts=1, prompt_len=200, fanout=2, seg_len=40)
    f, ids = _forest(s)
    leaves = [ids[x] for x in s.leaves]
    q = _queries(len(leaves), s.heads, 60)
    O, L = f.decode(leaves, q.to(DEV))
    Oh, Lh = f.decode_host(leaves, q)
    f.sync()
    assert _same(Oh, O.cpu()) and _same(Lh, L.cpu())
    q16 = _queries(16, s.heads, 61).to(DEV)
    O2, L2 = f.prefill([leaves[0]], [16], q16)
    O3 = torch.empty_like(q16)
    L3 = torch.empty(16, s.heads.num_q_heads, dtype=torch.float32, device=DEV)
    tp.tp_prefill(f.handle, [leaves[0]], [16], q16, O3, L3)
    f.sync()
    assert _same(O2.cpu(), O3.cpu()) and _same(L2.cpu(), L3.cpu())
    f.close()
