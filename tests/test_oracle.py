"""Pins for the CPU oracle: values that do not come from the oracle itself.

Each test is chosen so that a plausible slip in the oracle (a dropped scale,
the wrong GQA head, a log in the wrong base, a missing max term, a node left
off a path, a block handed out in the wrong order) fails at least one of them.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from conftest import golden


def bf16(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)


def rand_bf16(gen, *shape):
    return torch.randn(*shape, generator=gen, dtype=torch.float32).to(torch.bfloat16)


# --------------------------------------------------------------------------
# attention definition
# --------------------------------------------------------------------------
def test_two_token_hand_example():
    g = golden("two_token.json")
    o, lse = oracle.path_attention(bf16(g["q"]), bf16(g["k"]), bf16(g["v"]))
    np.testing.assert_allclose(o, np.asarray(g["O"]), rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse, np.asarray(g["LSE"]), rtol=0, atol=1e-14)


def _sdpa_reference(q, k, v):
    """torch's own fp64 SDPA over the flat path, KV heads expanded by
    contiguous GQA grouping (q-head h reads kv head h // g)."""
    hq = q.shape[0]
    n, hkv, d = k.shape
    g = hq // hkv
    qq = q.double()[None, :, None, :]                                     # [1][Hq][1][d]
    kk = k.double().permute(1, 0, 2).repeat_interleave(g, dim=0)[None]   # [1][Hq][N][d]
    vv = v.double().permute(1, 0, 2).repeat_interleave(g, dim=0)[None]
    o = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv)[0, :, 0, :]
    lse = torch.logsumexp((qq @ kk.transpose(-1, -2))[0, :, 0, :] / math.sqrt(d), dim=-1)
    return o.numpy(), lse.numpy()


@pytest.mark.parametrize("hq,hkv,d,n", [(1, 1, 16, 1), (4, 1, 64, 37), (8, 2, 64, 300),
                                        (28, 4, 128, 129), (6, 3, 32, 2)])
def test_matches_torch_sdpa(hq, hkv, d, n):
    gen = torch.Generator().manual_seed(hq * 1000 + n)
    q = rand_bf16(gen, hq, d)
    k = rand_bf16(gen, n, hkv, d) * 2          # wider score range
    v = rand_bf16(gen, n, hkv, d)
    o, lse = oracle.path_attention(q, k, v)
    o_ref, lse_ref = _sdpa_reference(q, k, v)
    np.testing.assert_allclose(o, o_ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse_ref, rtol=0, atol=1e-12)


def test_gqa_heads_are_contiguous_groups():
    # kv head c carries V = c+1 everywhere: q-head h must output h // g + 1.
    hq, hkv, d, n = 8, 4, 16, 5
    gen = torch.Generator().manual_seed(3)
    q = rand_bf16(gen, hq, d)
    k = rand_bf16(gen, n, hkv, d)
    v = torch.ones(n, hkv, d)
    for c in range(hkv):
        v[:, c, :] = c + 1
    o, _ = oracle.path_attention(q, k, v.to(torch.bfloat16))
    for h in range(hq):
        np.testing.assert_allclose(o[h], h // (hq // hkv) + 1, atol=1e-13)


def test_constant_values_give_that_value():
    gen = torch.Generator().manual_seed(4)
    q = rand_bf16(gen, 4, 64)
    k = rand_bf16(gen, 50, 2, 64)
    row = rand_bf16(gen, 2, 64)
    v = row[None].expand(50, 2, 64).contiguous()
    o, _ = oracle.path_attention(q, k, v)
    for h in range(4):
        np.testing.assert_allclose(o[h], row[h // 2].double().numpy(), atol=1e-13)


def test_zero_query_is_mean_and_log_n():
    gen = torch.Generator().manual_seed(5)
    n = 77
    q = torch.zeros(2, 32, dtype=torch.bfloat16)
    k = rand_bf16(gen, n, 1, 32)
    v = rand_bf16(gen, n, 1, 32)
    o, lse = oracle.path_attention(q, k, v)
    np.testing.assert_allclose(o[0], v[:, 0, :].double().mean(0).numpy(), atol=1e-13)
    np.testing.assert_allclose(lse, math.log(n), atol=1e-14)


def test_single_token_gives_its_value_and_score():
    # q = (1,2,0,...), k = (3,-1,0,...), d = 16: s = (3 - 2)/4 = 0.25
    d = 16
    q = torch.zeros(1, d)
    q[0, 0], q[0, 1] = 1, 2
    k = torch.zeros(1, 1, d)
    k[0, 0, 0], k[0, 0, 1] = 3, -1
    v = torch.arange(d, dtype=torch.float32).reshape(1, 1, d)
    o, lse = oracle.path_attention(q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16))
    np.testing.assert_array_equal(o[0], np.arange(d))
    assert lse[0] == 0.25


@pytest.mark.parametrize("order", [(0, 1, 2), (2, 1, 0), (2, 0, 1), (1, 2, 0), (2, 0)])
def test_large_scores_do_not_overflow(order):
    # scores ~ +-1000 (max in every position): exp would overflow unless the
    # true maximum is subtracted. Row i has score s_i and value e_i.
    q = bf16([[64.0, 0, 0, 0]])
    krows = [[[31.25, 0, 0, 0]], [[30.0, 0, 0, 0]], [[-31.25, 0, 0, 0]]]
    vrows = [[[1, 0, 0, 0]], [[0, 1, 0, 0]], [[0, 0, 1, 0]]]
    k = bf16([krows[i] for i in order])
    v = bf16([vrows[i] for i in order])
    o, lse = oracle.path_attention(q, k, v)
    s = {0: 1000.0, 1: 960.0, 2: -1000.0}
    top = max(s[i] for i in order)
    lse_ref = top + math.log(sum(math.exp(s[i] - top) for i in order))
    assert abs(lse[0] - lse_ref) < 1e-12
    expect = np.zeros(4)
    for i in order:
        expect[i] = math.exp(s[i] - lse_ref)
    np.testing.assert_allclose(o[0], expect, atol=1e-15)


def test_path_scores_hand_examples():
    # two-token golden: q = (2,0,0,0), d = 4, k_1 = 0, k_2 = e_1 -> s = (0, 1)
    g = golden("two_token.json")
    s = oracle.path_scores(bf16(g["q"]), bf16(g["k"]))
    np.testing.assert_array_equal(s, [[0.0, 1.0]])
    # q = (1,2,0,...), k = (3,-1,0,...), d = 16 -> s = (3 - 2) / 4
    q = torch.zeros(1, 16)
    q[0, 0], q[0, 1] = 1, 2
    k = torch.zeros(1, 1, 16)
    k[0, 0, 0], k[0, 0, 1] = 3, -1
    assert oracle.path_scores(q.to(torch.bfloat16), k.to(torch.bfloat16))[0, 0] == 0.25


@pytest.mark.parametrize("hq,hkv,d,n", [(4, 1, 64, 37), (28, 4, 128, 129), (6, 3, 32, 2)])
def test_path_scores_match_torch_and_give_the_oracle_lse(hq, hkv, d, n):
    # torch's fp64 product over the GQA-expanded path, and the C oracle's LSE
    # as the log-sum-exp of the scores (two independent routes)
    gen = torch.Generator().manual_seed(hq + 7 * n)
    q = rand_bf16(gen, hq, d)
    k = rand_bf16(gen, n, hkv, d) * 3
    v = rand_bf16(gen, n, hkv, d)
    s = oracle.path_scores(q, k)
    kk = k.double().permute(1, 0, 2).repeat_interleave(hq // hkv, dim=0)      # [Hq][N][d]
    ref = torch.einsum("hd,hnd->hn", q.double(), kk) / math.sqrt(d)
    np.testing.assert_allclose(s, ref.numpy(), rtol=0, atol=1e-12)
    _, lse = oracle.path_attention(q, k, v)
    np.testing.assert_allclose(torch.logsumexp(torch.from_numpy(s), dim=-1).numpy(), lse, rtol=0, atol=1e-12)


def test_path_scores_use_contiguous_gqa_groups():
    # kv head c holds k = (c+1) e_0, q = e_0: q-head h scores (h // g + 1) / sqrt(d)
    hq, hkv, d = 6, 3, 16
    q = torch.zeros(hq, d)
    q[:, 0] = 1
    k = torch.zeros(2, hkv, d)
    for c in range(hkv):
        k[:, c, 0] = c + 1
    s = oracle.path_scores(q.to(torch.bfloat16), k.to(torch.bfloat16))
    for h in range(hq):
        np.testing.assert_array_equal(s[h], (h // 2 + 1) / 4.0)


@pytest.mark.parametrize("cuts", [[1], [5, 64], [31, 32, 33, 200], list(range(1, 299, 7))])
def test_lse_merge_of_any_split_equals_whole(cuts):
    gen = torch.Generator().manual_seed(len(cuts))
    n = 299
    q = rand_bf16(gen, 8, 64)
    k = rand_bf16(gen, n, 2, 64)
    v = rand_bf16(gen, n, 2, 64)
    whole = oracle.path_attention(q, k, v)
    bounds = [0] + cuts + [n]
    parts = [oracle.path_attention(q, k[a:b], v[a:b]) for a, b in zip(bounds[:-1], bounds[1:])]
    merged = oracle.lse_merge(parts)
    np.testing.assert_allclose(merged[0], whole[0], rtol=0, atol=1e-12)
    np.testing.assert_allclose(merged[1], whole[1], rtol=0, atol=1e-12)


def test_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.path_attention(torch.zeros(3, 8, dtype=torch.bfloat16),
                              torch.zeros(4, 2, 8, dtype=torch.bfloat16),
                              torch.zeros(4, 2, 8, dtype=torch.bfloat16))   # 3 % 2 != 0


# --------------------------------------------------------------------------
# tree model: paths
# --------------------------------------------------------------------------
def _forward_paths(script):
    """Brute force, independent of parent walks: carry every live node's full
    kv_id list forward, copying it into each child at a fork."""
    path = {}
    for op in script.ops:
        if op[0] == "root":
            path[op[1]] = []
        elif op[0] == "append":
            path[op[1]] = path[op[1]] + [op[2]]
        elif op[0] == "fork":
            for c in op[2]:
                path[c] = list(path[op[1]])
    return path


@pytest.mark.parametrize("seed", range(6))
def test_paths_match_forward_construction(seed):
    s = workloads.random_tree(seed=seed, n_prompts=4, max_depth=5)
    model = oracle.OracleForest(block_tokens=16).replay(s)
    fwd = _forward_paths(s)
    for leaf in s.leaves:
        assert model.path_chunks(leaf) == fwd[leaf]


@pytest.mark.parametrize("name", ["tiny", "qwen7b", "random_divergence", "wide_prefix", "no_sharing"])
def test_named_workload_shapes(name):
    small = {"tiny": {}, "qwen7b": {"n_prompts": 3}, "random_divergence": {"n_prompts": 3},
             "wide_prefix": {"n_prompts": 1}, "no_sharing": {"n_seqs": 3}}[name]
    s = workloads.by_name(name, **small)
    model = oracle.OracleForest(block_tokens=32).replay(s)
    fwd = _forward_paths(s)
    lens = {lf: sum(s.kv_len[c] for c in fwd[lf]) for lf in s.leaves}
    if name == "tiny":
        assert len(s.leaves) == 8
        assert all(193 <= n <= 224 for n in lens.values())
    elif name == "qwen7b":
        assert len(s.leaves) == 3 * 16
        assert all(256 + 2048 <= n <= 1024 + 2048 for n in lens.values())
    elif name == "random_divergence":
        assert all(n == 1024 + 14 * 512 for n in lens.values())
    elif name == "wide_prefix":
        assert len(s.leaves) == 64 and set(lens.values()) == {2048 + 5 * 256}
    else:
        assert set(lens.values()) == {4096}
    for lf in s.leaves:
        assert model.path_chunks(lf) == fwd[lf]


def test_random_divergence_full_size_statistics():
    # Seeded reading of the growth rule reproduces the intended scale:
    # ~940 leaves, ~3.3 M unique path tokens, sharing ratio ~2.3.
    s = workloads.random_divergence(seed=0)
    model = oracle.OracleForest(block_tokens=32, pool_blocks=1 << 19).replay(s)
    n = len(s.leaves)
    uniq = model.unique_path_tokens(s.leaves)
    assert n == 940
    assert 3.2e6 < uniq < 3.5e6
    assert 2.2 < n * 8192 / uniq < 2.4


# --------------------------------------------------------------------------
# tree model: pool
# --------------------------------------------------------------------------
def test_block_allocation_golden():
    g = golden("block_allocation.json")
    m = oracle.OracleForest(block_tokens=g["block_tokens"], pool_blocks=g["pool_blocks"])

    def apply(op):
        if op[0] == "root":
            m.add_root(op[1])
        elif op[0] == "append":
            m.append(op[1], op[2], op[3])
        elif op[0] == "fork":
            m.fork(op[1], op[2])
        elif op[0] == "prune":
            m.prune(op[1])

    for step in g["steps"]:
        if "op" in step:
            apply(step["op"])
        elif "check_path" in step:
            leaf, slots = step["check_path"]
            assert m.path_slots(leaf).tolist() == slots, step
        elif "check_live_blocks" in step:
            assert m.live_blocks() == step["check_live_blocks"]
        elif "expect_error" in step:
            with pytest.raises(oracle.OracleError) as e:
                apply(step["expect_error"])
            assert e.value.code == step["code"]


@pytest.mark.parametrize("seed", range(4))
def test_pool_invariants(seed):
    s = workloads.random_tree(seed=seed, n_prompts=5, max_depth=5, p_prune=0.35)
    bt = 8
    m = oracle.OracleForest(block_tokens=bt, pool_blocks=4096).replay(s)
    owned = []
    for nid, node in m.nodes.items():
        if node.state == "dead":
            assert node.blocks == []
            continue
        assert len(node.blocks) == -(-node.n_tokens // bt)
        owned += node.blocks
    assert len(owned) == len(set(owned)) == m.live_blocks()
    # every live token has its own slot; shared prefixes give shared slots
    for lf in set(s.leaves):
        sl = m.path_slots(lf)
        assert len(sl) == len(set(sl.tolist()))
        assert len(sl) == sum(m.kv_len[c] for c in m.path_chunks(lf))


# --------------------------------------------------------------------------
# whole oracle decode
# --------------------------------------------------------------------------
def test_forest_decode_matches_sdpa_on_flat_paths():
    s = workloads.random_tree(seed=11, n_prompts=3, max_depth=4, heads=workloads.Heads(8, 2, 32))
    m = oracle.OracleForest(block_tokens=16).replay(s)
    q = s.q()
    o, lse = m.decode(s.leaves, q, s.kv, threads=4)
    fwd = _forward_paths(s)
    for i, lf in enumerate(s.leaves):
        kvs = [s.kv(c) for c in fwd[lf]]
        k = torch.cat([a for a, _ in kvs])
        v = torch.cat([b for _, b in kvs])
        o_ref, lse_ref = _sdpa_reference(q[i], k, v)
        np.testing.assert_allclose(o[i], o_ref, atol=1e-12)
        np.testing.assert_allclose(lse[i], lse_ref, atol=1e-12)


def test_single_branch_equals_last_row_of_causal_attention():
    s = workloads.single_path(seed=2, lengths=(40, 33, 1, 60), heads=workloads.Heads(4, 2, 64))
    m = oracle.OracleForest(block_tokens=32).replay(s)
    q = s.q()
    o, lse = m.decode(s.leaves, q, s.kv)
    k = torch.cat([s.kv(c)[0] for c in range(len(s.kv_len))])
    v = torch.cat([s.kv(c)[1] for c in range(len(s.kv_len))])
    n = k.shape[0]
    gen = torch.Generator().manual_seed(9)
    qs = torch.randn(n, 4, 64, generator=gen, dtype=torch.float64)
    qs[-1] = q[0].double()
    kk = k.double().permute(1, 0, 2).repeat_interleave(2, dim=0)[None]
    vv = v.double().permute(1, 0, 2).repeat_interleave(2, dim=0)[None]
    causal = torch.nn.functional.scaled_dot_product_attention(qs.permute(1, 0, 2)[None], kk, vv, is_causal=True)
    np.testing.assert_allclose(o[0], causal[0, :, -1, :].numpy(), atol=1e-12)


def test_identical_paths_and_queries_are_bitwise_identical():
    # two sibling leaves that received the same K/V, and one leaf listed twice
    s = workloads.tiny(seed=1)
    m = oracle.OracleForest(block_tokens=32).replay(s)
    a, b = s.leaves[0], s.leaves[1]
    last_a = m.nodes[a].chunks[-1]

    def same_kv(kv_id):
        return s.kv(last_a if kv_id == m.nodes[b].chunks[-1] else kv_id)

    q1 = s.q(n=1)[0]
    q = torch.stack([q1, q1, q1])
    o, lse = m.decode([a, b, a], q, same_kv, threads=1)
    assert np.array_equal(o[0], o[1]) and np.array_equal(o[0], o[2])
    assert np.array_equal(lse[0], lse[1]) and np.array_equal(lse[0], lse[2])


def test_empty_path_is_rejected():
    m = oracle.OracleForest(block_tokens=32)
    m.add_root(0)
    with pytest.raises(oracle.OracleError) as e:
        m.decode([0], torch.zeros(1, 1, 8, dtype=torch.bfloat16), lambda i: None)
    assert e.value.code == "EMPTY_PATH"


# --------------------------------------------------------------------------
# prefill (causal multi-query attention)
# --------------------------------------------------------------------------
def _causal_sdpa_rows(k, v, qrows, first_pos, group):
    """torch fp64 SDPA with an explicit mask: query r (at path position
    first_pos + r) sees positions <= its own."""
    n = k.shape[0]
    m = qrows.shape[0]
    kk = k.double().permute(1, 0, 2).repeat_interleave(group, dim=0)[None]
    vv = v.double().permute(1, 0, 2).repeat_interleave(group, dim=0)[None]
    qq = qrows.double().permute(1, 0, 2)[None]
    pos = torch.arange(n)[None, :]
    qpos = (first_pos + torch.arange(m))[:, None]
    mask = pos <= qpos
    o = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, attn_mask=mask)
    return o[0].permute(1, 0, 2).numpy()


def test_prefill_of_single_path_is_causal_sdpa():
    # one node path of 4 appended chunks; the whole last chunk and then every
    # token are queries: rows of torch's causal attention
    s = workloads.single_path(seed=3, lengths=(37, 20, 5, 41), heads=workloads.Heads(6, 2, 64))
    m = oracle.OracleForest(block_tokens=32).replay(s)
    leaf = s.leaves[0]
    k = torch.cat([s.kv(c)[0] for c in range(len(s.kv_len))])
    v = torch.cat([s.kv(c)[1] for c in range(len(s.kv_len))])
    n = k.shape[0]
    node_tokens = m.nodes[leaf].n_tokens
    gen = torch.Generator().manual_seed(4)
    for mq in (1, 7, node_tokens):
        q = torch.randn(mq, 6, 64, generator=gen).to(torch.bfloat16)
        o, lse = m.prefill([leaf], [mq], q, s.kv)
        ref = _causal_sdpa_rows(k, v, q, n - mq, 3)
        np.testing.assert_allclose(o, ref, atol=1e-12)


def test_prefill_on_tree_matches_flat_causal_attention_per_node():
    s = workloads.random_tree(seed=5, n_prompts=2, max_depth=4, heads=workloads.Heads(8, 2, 32))
    m = oracle.OracleForest(block_tokens=16).replay(s)
    fwd = _forward_paths(s)
    live = [x for x, nd in m.nodes.items() if nd.state != "dead" and nd.n_tokens > 0]
    nodes = live[:6]
    counts = [min(m.nodes[x].n_tokens, 1 + (3 * i) % 9) for i, x in enumerate(nodes)]
    gen = torch.Generator().manual_seed(6)
    q = torch.randn(sum(counts), 8, 32, generator=gen).to(torch.bfloat16)
    o, lse = m.prefill(nodes, counts, q, s.kv, threads=4)
    r = 0
    for x, mq in zip(nodes, counts):
        chunks = [c for y in m.path_nodes(x, True) for c in m.nodes[y].chunks]
        k = torch.cat([s.kv(c)[0] for c in chunks])
        v = torch.cat([s.kv(c)[1] for c in chunks])
        ref = _causal_sdpa_rows(k, v, q[r:r + mq], k.shape[0] - mq, 4)
        np.testing.assert_allclose(o[r:r + mq], ref, atol=1e-12)
        r += mq
    assert r == len(q) and np.isfinite(lse).all()


def test_prefill_of_last_token_equals_decode():
    s = workloads.tiny(seed=2)
    m = oracle.OracleForest(block_tokens=32).replay(s)
    q = s.q()
    o_d, lse_d = m.decode(s.leaves, q, s.kv)
    o_p, lse_p = m.prefill(s.leaves, [1] * len(s.leaves), q, s.kv)
    np.testing.assert_array_equal(o_d, o_p)
    np.testing.assert_array_equal(lse_d, lse_p)
