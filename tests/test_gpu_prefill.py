"""GPU parity of tp_prefill (causal multi-query attention over tree paths)
against the oracle's prefill -- the decode definition applied to each prefix
of each path. Tolerances as in test_gpu_parity (contract bar and the
2^-8 (|O| + A) + 1e-5 rounding bar, |dLSE| <= 5e-5)."""
import numpy as np
import pytest
import torch

import oracle
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


def _src(script):
    cache = {}

    def src(kv_id):
        if kv_id not in cache:
            k, v = script.kv(kv_id, DEV)
            cache[kv_id] = (k.cpu(), v.cpu())
        return cache[kv_id]
    return src


def run_prefill(script, nodes_sid, counts, rows=None, seed=0, flags=0, o_offset=0):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=script.upper_bound_blocks(32) + 64,
                  device=DEV)
    ids = f.replay(script.ops, kv_fn=lambda kv_id: script.kv(kv_id, DEV))
    total = sum(counts)
    g = torch.Generator(device="cpu").manual_seed(seed)
    Q = torch.randn(total, h.num_q_heads, h.head_dim, generator=g).to(torch.bfloat16).to(DEV)
    # o_offset elements into a larger buffer: an O that is 16-byte but not
    # 32-byte aligned takes the kernel's 16-byte store path
    O_buf = torch.empty(Q.numel() + o_offset, dtype=torch.bfloat16, device=DEV)
    O = O_buf[o_offset:].view(Q.shape)
    LSE = torch.empty(total, h.num_q_heads, dtype=torch.float32, device=DEV)
    tp.tp_prefill(f.handle, [ids[x] for x in nodes_sid], counts, Q, O, LSE, flags)
    f.sync()
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(script)
    src = _src(script)
    o_ref, lse_ref = model.prefill(nodes_sid, counts, Q.cpu(), src, indices=rows)

    def abs_src(kv_id):
        k, v = src(kv_id)
        return k, oracle.bf16_bits(v) & np.uint16(0x7FFF)
    a_ref, _ = model.prefill(nodes_sid, counts, Q.cpu(), abs_src, indices=rows)
    sel = list(range(total)) if rows is None else sorted(rows)
    o = O.float().cpu().numpy().astype(np.float64)[sel]
    lse = LSE.cpu().numpy().astype(np.float64)[sel]
    o_ref, lse_ref, a_ref = o_ref[sel], lse_ref[sel], a_ref[sel]
    d_o, d_lse = np.abs(o - o_ref), np.abs(lse - lse_ref)
    assert np.isfinite(o).all() and np.isfinite(lse).all()
    assert d_o.max() <= 1e-2 and d_lse.max() <= 1e-3, (d_o.max(), d_lse.max())
    assert (d_o - (2.0 ** -8 * (np.abs(o_ref) + a_ref) + 1e-5)).max() <= 0, d_o.max()
    assert d_lse.max() <= 5e-5, d_lse.max()
    f.close()
    return O, LSE


FLAGS = [0, tp.TP_MMA_SYNC]


@pytest.mark.parametrize("flags", FLAGS)
@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("heads", [workloads.Heads(8, 2, 64), workloads.Heads(28, 4, 128)])
def test_prefill_random_trees(seed, heads, flags):
    s = workloads.random_tree(seed=seed, n_prompts=3, max_depth=4, heads=heads)
    model = oracle.OracleForest(block_tokens=32).replay(s)
    rng = np.random.default_rng(seed)
    live = [x for x in model.nodes if model.nodes[x].state != "dead" and model.nodes[x].n_tokens > 0]
    pick = [live[int(i)] for i in rng.integers(0, len(live), min(len(live), 8))]
    counts = [int(rng.integers(0, model.nodes[x].n_tokens + 1)) for x in pick]
    if sum(counts) == 0:
        counts[0] = 1
    run_prefill(s, pick, counts, seed=seed, flags=flags)


@pytest.mark.parametrize("flags", FLAGS)
def test_prefill_whole_segments_of_a_wide_tree(flags):
    # 4 prompts of 1024 tokens, each forked into 4 leaves holding 512-token
    # segments; every leaf's whole segment is a query block (8192 queries)
    s = workloads.segment_prefill(seed=2, n_prompts=4, prompt_len=1024, fanout=4, seg_len=512)
    counts = [512] * len(s.leaves)
    rng = np.random.default_rng(0)
    total = sum(counts)
    rows = sorted(set([0, 511, 512, total - 1] + [int(x) for x in rng.integers(0, total, 96)]))
    run_prefill(s, list(s.leaves), counts, rows=rows, flags=flags)


@pytest.mark.parametrize("flags", FLAGS)
def test_prefill_long_path_several_chunks(flags):
    # 5000-token prompt and a 700-token segment: row blocks need several
    # chunks (partials + merge) next to single-chunk blocks (direct output)
    s = workloads.single_path(seed=4, lengths=(5000, 700), heads=workloads.Heads(28, 4, 128))
    rng = np.random.default_rng(1)
    rows = sorted(set([0, 1, 699] + [int(x) for x in rng.integers(0, 700, 60)]))
    run_prefill(s, list(s.leaves), [700], rows=rows, flags=flags)


@pytest.mark.parametrize("flags", FLAGS)
def test_prefill_output_16_byte_aligned_only(flags):
    # the wide-tree case again (its row blocks write O directly and through
    # the merge), with O 16 bytes past a 32-byte boundary
    s = workloads.segment_prefill(seed=2, n_prompts=4, prompt_len=1024, fanout=4, seg_len=512)
    counts = [512] * len(s.leaves)
    total = sum(counts)
    rng = np.random.default_rng(3)
    rows = sorted(set([0, 511, 512, total - 1] + [int(x) for x in rng.integers(0, total, 64)]))
    O, _ = run_prefill(s, list(s.leaves), counts, rows=rows, o_offset=8, flags=flags)
    assert O.data_ptr() % 32 == 16


def test_prefill_last_token_matches_decode():
    s = workloads.tiny(seed=3)
    h = s.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=s.upper_bound_blocks(32) + 8, device=DEV)
    ids = f.replay(s.ops, kv_fn=lambda kv_id: s.kv(kv_id, DEV))
    leaves = [ids[x] for x in s.leaves]
    Q = s.q(DEV)
    O1, L1 = f.decode(leaves, Q)
    O2 = torch.empty_like(Q)
    L2 = torch.empty_like(L1)
    tp.tp_prefill(f.handle, leaves, [1] * len(leaves), Q, O2, L2)
    f.sync()
    assert (O1.float() - O2.float()).abs().max().item() <= 2 ** -7
    assert (L1 - L2).abs().max().item() <= 5e-5
    f.close()


@pytest.mark.parametrize("seed", range(100, 112))
def test_prefill_random_sweep(seed):
    rng = np.random.default_rng(seed)
    heads = [workloads.Heads(8, 2, 64), workloads.Heads(28, 4, 128), workloads.Heads(64, 8, 128),
             workloads.Heads(16, 16, 128)][seed % 4]
    s = workloads.random_tree(seed=seed, n_prompts=int(rng.integers(1, 4)), max_depth=int(rng.integers(1, 6)),
                              heads=heads, prompt_range=(1, int(rng.integers(2, 600))),
                              seg_range=(1, int(rng.integers(2, 300))))
    model = oracle.OracleForest(block_tokens=32).replay(s)
    live = [x for x in model.nodes if model.nodes[x].state != "dead" and model.nodes[x].n_tokens > 0]
    pick = [live[int(i)] for i in rng.integers(0, len(live), min(len(live), 10))]
    counts = [int(rng.integers(0, model.nodes[x].n_tokens + 1)) for x in pick]
    if sum(counts) == 0:
        counts[0] = 1
    run_prefill(s, pick, counts, seed=seed, flags=FLAGS[seed % 2])


def test_prefill_back_to_back_calls_and_decode_cache():
    # Prefill schedules go to two device buffers used in turn, each uploaded
    # on a copy stream once the call two back has finished reading it. Four
    # calls of growing and shrinking size are issued with no sync between
    # them (both buffers grow while the other call is in flight), between two
    # decode calls of the same leaves; the second decode reuses the cached
    # decode schedule, which prefill no longer touches, and gives the same
    # bits as the first.
    s = workloads.random_tree(seed=7, n_prompts=3, max_depth=4, heads=workloads.Heads(28, 4, 128))
    h = s.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=s.upper_bound_blocks(32) + 64, device=DEV)
    ids = f.replay(s.ops, kv_fn=lambda kv_id: s.kv(kv_id, DEV))
    leaves = [ids[x] for x in s.leaves]
    Qd = s.q(DEV)
    O1, L1 = f.decode(leaves, Qd)
    model = oracle.OracleForest(block_tokens=32, pool_blocks=f.cfg.pool_blocks).replay(s)
    live = [x for x in model.nodes if model.nodes[x].state != "dead" and model.nodes[x].n_tokens > 0]
    rng = np.random.default_rng(7)
    calls = []
    for n_pick, frac in ((2, 0.2), (8, 1.0), (1, 0.1), (10, 1.0)):
        pick = [live[int(i)] for i in rng.integers(0, len(live), min(len(live), n_pick))]
        counts = [max(1, int(frac * model.nodes[x].n_tokens)) for x in pick]
        g = torch.Generator(device="cpu").manual_seed(len(calls))
        Q = torch.randn(sum(counts), h.num_q_heads, h.head_dim, generator=g).to(torch.bfloat16).to(DEV)
        O, LSE = torch.empty_like(Q), torch.empty(Q.shape[:2], dtype=torch.float32, device=DEV)
        tp.tp_prefill(f.handle, [ids[x] for x in pick], counts, Q, O, LSE, 0)
        calls.append((pick, counts, Q, O, LSE))
    O2, L2 = f.decode(leaves, Qd)
    f.sync()
    assert torch.equal(O1, O2) and torch.equal(L1, L2)
    src = _src(s)
    for pick, counts, Q, O, LSE in calls:
        total = sum(counts)
        rows = sorted(set([0, total - 1] + [int(x) for x in rng.integers(0, total, 48)]))
        o_ref, lse_ref = model.prefill(pick, counts, Q.cpu(), src, indices=rows)
        o = O.float().cpu().numpy().astype(np.float64)[rows]
        lse = LSE.cpu().numpy().astype(np.float64)[rows]
        assert np.abs(o - o_ref[rows]).max() <= 1e-2
        assert np.abs(lse - lse_ref[rows]).max() <= 5e-5
    f.close()
