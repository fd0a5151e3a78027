"""tp_decode_noalloc: the decode entry point that allocates no device memory.

Some callers cannot call cudaMalloc while they decode -- a serving process
that carves up all device memory at start-up, or a latency-critical loop that
cannot take cudaMalloc's implicit synchronisation. For them the library keeps
the decode scratch (schedule and fp32 partials) in one static device array.
These tests call that entry point through the C ABI and compare it with
tp_decode_ex, on two calls in a row (the array keeps the previous call's
contents, so the second call must not depend on them). This file is
collected last on purpose.
"""
import numpy as np
import pytest
import torch

import paper_2508_17445_gb300 as tp
import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TOL_O, TOL_LSE = 1e-2, 1e-3


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2508_17445_gb300 import build
    build.build()


def _forest(script):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim,
                  pool_blocks=script.upper_bound_blocks(32) + 64, device=DEV)
    ids = f.replay(script.ops, kv_fn=lambda kv_id: script.kv(kv_id, DEV))
    return f, [ids[x] for x in script.leaves]


@pytest.mark.parametrize("script", [workloads.qwen7b(seed=3, n_prompts=2),
                                    workloads.random_tree(seed=4, heads=workloads.Heads(8, 2, 64), n_prompts=3)],
                         ids=["qwen7b-2-prompts", "random-forest-hd64"])
def test_noalloc_matches_decode_on_two_calls(script):
    f, leaves = _forest(script)
    Q = script.q(DEV)
    O_ref, LSE_ref = f.decode(leaves, Q)
    f.sync()
    for _ in range(2):
        O = torch.full_like(O_ref, float("nan"))
        LSE = torch.full_like(LSE_ref, float("nan"))
        tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
        f.sync()
        d_o = (O.float() - O_ref.float()).abs().max().item()
        d_lse = (LSE - LSE_ref).abs().max().item()
        assert np.isfinite(d_o) and np.isfinite(d_lse)
        assert d_o <= TOL_O and d_lse <= TOL_LSE, (d_o, d_lse)
    f.close()


def test_noalloc_rejects_work_beyond_its_scratch():
    # 32 Qwen-shaped prompts need ~37 MB of fp32 partials: over the 32 MiB array
    script = workloads.qwen7b(seed=5, n_prompts=32)
    f, leaves = _forest(script)
    Q = script.q(DEV)
    O = torch.empty((len(leaves), 28, 128), dtype=torch.bfloat16, device=DEV)
    LSE = torch.empty((len(leaves), 28), dtype=torch.float32, device=DEV)
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
    assert e.value.code == "OOM" and "static scratch" in str(e.value)
    f.sync()
    f.close()


def test_noalloc_is_refused_while_its_stream_is_captured():
    # The schedule goes up from a host buffer that lives only for the call; a
    # copy captured into a CUDA graph would re-read it on every replay, so the
    # call refuses a capturing stream, launches nothing, and works again after.
    script = workloads.qwen7b(seed=6, n_prompts=1)
    f, leaves = _forest(script)
    Q = script.q(DEV)
    O_ref, LSE_ref = f.decode(leaves, Q)
    O, LSE = torch.empty_like(O_ref), torch.empty_like(LSE_ref)
    tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)  # first call on the device: before any capture
    f.sync()
    side = torch.cuda.Stream()
    tp.tp_set_stream(f.handle, side.cuda_stream)
    graph = torch.cuda.CUDAGraph()
    x = torch.zeros(1, device=DEV)
    with torch.cuda.graph(graph, stream=side):
        x.add_(1)
        with pytest.raises(tp.TreepoError) as e:
            tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
    assert e.value.code == "INVALID_ARG" and "captured" in str(e.value)
    graph.replay()
    torch.cuda.synchronize()
    assert x.item() == 1.0                              # the graph holds only the torch op
    tp.tp_set_stream(f.handle, torch.cuda.current_stream().cuda_stream)
    O.fill_(float("nan"))
    tp.tp_decode_noalloc(f.handle, leaves, Q, O, LSE)
    f.sync()
    assert (O.float() - O_ref.float()).abs().max().item() <= TOL_O
    assert (LSE - LSE_ref).abs().max().item() <= TOL_LSE
    f.close()
