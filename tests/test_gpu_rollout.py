"""GPU parity of the sampler side of the library: the stand-in activations,
the decode loop (one-token appends with the cached schedule patched in
place), a whole Algorithm 1 rollout with decode after every token, and the
tree advantage kernel -- each against the CPU oracles.

Attention tolerances are those of test_gpu_parity: the contract bar
(|dO| <= 1e-2, |dLSE| <= 1e-3) and the rounding bar |dO| <= 2^-8 (|O| + A)
+ 1e-5, |dLSE| <= 5e-5 with A the attention output over |V|. The advantage
is accumulated in fp64 and stored as fp32: |d adv| <= 1e-6 (|adv| + 1).
"""
import numpy as np
import pytest
import torch

import oracle
import oracle.advantage as OA
import oracle.rollout as R
import paper_2508_17445_gb300 as tp
from conftest import golden

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2508_17445_gb300 import build
    build.build()


def bits_tensor(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16)


def oracle_attention(q_bits, k_bits, v_bits):
    o, lse = oracle.path_attention(q_bits, k_bits, v_bits)
    a, _ = oracle.path_attention(q_bits, k_bits, v_bits & np.uint16(0x7FFF))
    return o, lse, a


def check_rows(o_gpu, lse_gpu, refs):
    o = o_gpu.float().cpu().numpy().astype(np.float64)
    lse = lse_gpu.cpu().numpy().astype(np.float64)
    for i, (o_ref, lse_ref, a_ref) in enumerate(refs):
        d_o, d_lse = np.abs(o[i] - o_ref), np.abs(lse[i] - lse_ref)
        assert d_o.max() <= 1e-2 and d_lse.max() <= 1e-3, (i, d_o.max(), d_lse.max())
        assert (d_o - (2.0 ** -8 * (np.abs(o_ref) + a_ref) + 1e-5)).max() <= 0, (i, d_o.max())
        assert d_lse.max() <= 5e-5, (i, d_lse.max())


# ---------------------------------------------------------- activations --
@pytest.mark.parametrize("heads", [(28, 4, 128), (8, 2, 64)])
def test_synth_tokens_bit_exact(heads):
    hq, hkv, hd = heads
    f = tp.Forest(hq, hkv, hd, pool_blocks=4, device=DEV)
    for seed, node, pos0, n in ((0, 0, 0, 37), (2 ** 63 + 5, 12345, 1000, 300), (7, (1 << 28) - 1, (1 << 20) - 9, 9)):
        K = torch.empty((n, hkv, hd), dtype=torch.bfloat16, device=DEV)
        V = torch.empty_like(K)
        Q = torch.empty((n, hq, hd), dtype=torch.bfloat16, device=DEV)
        tp.tp_synth_tokens(f.handle, seed, node, pos0, n, K, V, Q)
        f.sync()
        pos = list(range(pos0, pos0 + n))
        for t, tag, h in ((K, R.TAG_K, hkv), (V, R.TAG_V, hkv), (Q, R.TAG_Q, hq)):
            want = R.synth_rows(seed, tag, [node] * n, pos, h, hd)
            np.testing.assert_array_equal(oracle.bf16_bits(t), want)
    with pytest.raises(tp.TreepoError):
        tp.tp_synth_tokens(f.handle, 0, 1 << 28, 0, 1, None, None, None)
    f.close()


# ----------------------------------------------------------- decode loop --
def test_decode_loop_patched_schedule_matches_rebuild_and_oracle():
    """A prompt forked into paths that grow one token per step: every step's
    decode (schedule patched in place) must equal a from-scratch schedule's
    bit for bit, and the oracle within tolerance."""
    hq, hkv, hd = 8, 2, 64
    g = torch.Generator(device="cpu").manual_seed(3)
    rnd = lambda *s: torch.randn(*s, generator=g).to(torch.bfloat16)
    f = tp.Forest(hq, hkv, hd, pool_blocks=256, device=DEV)
    root = f.add_root()
    pk, pv = rnd(45, hkv, hd), rnd(45, hkv, hd)
    f.append(root, pk.to(DEV), pv.to(DEV))
    mid = f.fork(root, 2)
    hist = {}
    for m in mid:                                  # two shared segments of 20 tokens
        k, v = rnd(20, hkv, hd), rnd(20, hkv, hd)
        f.append(m, k.to(DEV), v.to(DEV))
        hist[m] = (k, v)
    leaves = []
    for m in mid:
        leaves += f.fork(m, 3)
    path_k = {x: [pk, hist[mid[i // 3]][0]] for i, x in enumerate(leaves)}
    path_v = {x: [pv, hist[mid[i // 3]][1]] for i, x in enumerate(leaves)}
    for step in range(75):
        K, V = rnd(len(leaves), hkv, hd), rnd(len(leaves), hkv, hd)
        f.append_tokens(leaves, K.to(DEV), V.to(DEV))
        for i, x in enumerate(leaves):
            path_k[x].append(K[i:i + 1])
            path_v[x].append(V[i:i + 1])
        Q = rnd(len(leaves), hq, hd).to(DEV)
        O1, L1 = f.decode(leaves, Q)
        O2, L2 = f.decode(leaves, Q, flags=tp.TP_DECODE_NO_CACHE)
        f.sync()
        assert torch.equal(O1.view(torch.int16), O2.view(torch.int16)) and torch.equal(L1, L2), step
        if step in (0, 1, 30, 31, 32, 74):
            refs = []
            for i, x in enumerate(leaves):
                kb = oracle.bf16_bits(torch.cat(path_k[x]))
                vb = oracle.bf16_bits(torch.cat(path_v[x]))
                refs.append(oracle_attention(oracle.bf16_bits(Q[i].cpu()), kb, vb))
            check_rows(O1, L1, refs)
        if step == 40:                             # a prune invalidates the cache structurally
            f.prune(leaves[-1])
            leaves.pop()
    f.close()


# -------------------------------------------------------------- rollout --
def rollout_pair(op: R.RolloutParams, heads, decode_flags=0, probe_calls=()):
    hq, hkv, hd = heads
    f = tp.Forest(hq, hkv, hd, pool_blocks=1 << 15, device=DEV)
    kw = dict(width=op.width, max_depth=op.max_depth, seg_tokens=op.seg_tokens, arity=op.arity,
              init_branches=op.init_branches, policy=op.policy, fallback=int(op.fallback),
              temperature=op.temperature, p_eos=op.p_eos, p_boxed=op.p_boxed, p_fail=op.p_fail,
              p_correct=op.p_correct, seed=op.seed, decode=1, decode_flags=decode_flags)
    params = tp.rollout_params(list(op.prompt_tokens), **kw)
    probes = []
    for call in probe_calls:
        cap = len(op.prompt_tokens) * op.width
        pr = dict(o=torch.zeros((cap, hq, hd), dtype=torch.bfloat16, device=DEV),
                  lse=torch.zeros((cap, hq), dtype=torch.float32, device=DEV),
                  rows=np.zeros((cap, 2), dtype=np.int32), n=np.zeros(1, dtype=np.int32))
        pr["struct"] = tp.TpRolloutProbe(call=call, cap=cap, o=pr["o"].data_ptr(), lse=pr["lse"].data_ptr(),
                                         rows=pr["rows"].ctypes.data, n_rows=pr["n"].ctypes.data)
        probes.append(pr)
    results = []
    for pr in probes or [None]:
        ev, st = f.rollout(params, probe=None if pr is None else pr["struct"])
        f.sync()
        results.append((ev, st))
    return f, results, probes


@pytest.mark.parametrize("heads,flags", [((8, 2, 64), 0), ((28, 4, 128), 0), ((8, 2, 64), tp.TP_DECODE_CUDA_CORE_SMALL)])
def test_rollout_with_decode_matches_oracle(heads, flags):
    op = R.RolloutParams(prompt_tokens=[70, 33, 96], width=8, max_depth=4, seg_tokens=40, arity=2,
                         init_branches=2, p_eos=1 / 64, p_boxed=0.15, p_fail=0.1, seed=21)
    res = R.rollout(op)
    want = R.events_array(res)
    probe_calls = (0, 39, 75, 118)
    f, results, probes = rollout_pair(op, heads, flags, probe_calls)
    hq, hkv, hd = heads
    first = f.node_info(0)
    for (ev, st), pr, call in zip(results, probes, probe_calls):
        # each rollout adds its roots after the previous one's nodes
        base = int(ev[0, 2])
        shifted = R.rollout(op, first_node=base)
        np.testing.assert_array_equal(ev, R.events_array(shifted))
        assert st["decode_calls"] > max(probe_calls) and st["decode_rows"] >= st["tokens"]
        n = int(pr["n"][0])
        assert n > 0
        refs = []
        for leaf, t in pr["rows"][:n]:
            kb, vb = R.path_kv(shifted, op.seed, int(leaf), int(t) + 1, hkv, hd)
            qb = R.synth_rows(op.seed, R.TAG_Q, [int(leaf)], [int(t)], hq, hd)[0]
            refs.append(oracle_attention(qb, kb.reshape(-1, hkv, hd), vb.reshape(-1, hkv, hd)))
        check_rows(pr["o"][:n], pr["lse"][:n], refs)
    assert f.stats()["live_nodes"] == 0 and f.stats()["free_blocks"] == f.stats()["pool_blocks"]
    assert first["parent"] == -1
    f.close()


def test_rollout_decode_and_dry_runs_agree_at_paper_shape():
    # 16 prompts, w = 16, 6 x 128 segments, log-prob branching (T = 2)
    op = R.RolloutParams(prompt_tokens=[int(x) for x in np.random.default_rng(5).integers(256, 1024, 16)],
                         width=16, max_depth=6, seg_tokens=128, init_branches=0, policy=R.BRANCH_LOGP_HIGH,
                         p_eos=1 / 1024, p_boxed=0.05, p_fail=0.05, seed=8)
    f, results, _ = rollout_pair(op, (28, 4, 128))
    ev, st = results[0]
    np.testing.assert_array_equal(ev, R.events_array(R.rollout(op)))
    dry = tp.Forest(28, 4, 128, pool_blocks=1 << 15, device=None)
    kw = dict(width=16, max_depth=6, seg_tokens=128, init_branches=0, policy=R.BRANCH_LOGP_HIGH,
              p_eos=1 / 1024, p_boxed=0.05, p_fail=0.05, seed=8)
    ev2, st2 = dry.rollout(tp.rollout_params(list(op.prompt_tokens), **kw))
    np.testing.assert_array_equal(ev, ev2)
    assert st["segments"] == st2["segments"] and st["decode_calls"] > 0
    f.close()


# ------------------------------------------------------------ advantage --
def run_advantage(parent, leaves, rewards):
    P = torch.tensor(parent, dtype=torch.int32, device=DEV)
    L = torch.tensor(leaves, dtype=torch.int32, device=DEV)
    Rw = torch.tensor(rewards, dtype=torch.float32, device=DEV)
    adv = torch.full((len(leaves),), 123.0, dtype=torch.float32, device=DEV)
    stats = torch.zeros(4, dtype=torch.float64, device=DEV)
    tp.tp_tree_advantage(P, L, Rw, adv, stats)
    torch.cuda.synchronize()
    return adv.cpu().numpy().astype(np.float64), stats.cpu().numpy()


def check_advantage(parent, leaves, rewards):
    adv, stats = run_advantage(parent, leaves, rewards)
    want, st = OA.tree_advantage(parent, leaves, np.asarray(rewards, dtype=np.float32).astype(np.float64))
    assert np.all(np.abs(adv - want) <= 1e-6 * (np.abs(want) + 1)), np.abs(adv - want).max()
    assert stats[0] == st["accepted"] and abs(stats[2] - st["std"]) <= 1e-12 * (1 + st["std"]) and stats[3] == 0
    return adv


def test_advantage_hand_example():
    g = golden("tree_advantage_figure.json")
    adv = check_advantage(g["parent"], g["leaves"], g["rewards"])
    a = np.array(g["A_times_3"]) / 3
    np.testing.assert_allclose(adv, a / np.sqrt(g["std_squared_times_9"] / 9), rtol=1e-6)


def random_forest(rng, n_roots, n_nodes):
    """Random forest with parents drawn among earlier nodes, then relabelled
    so that ids do not follow creation order."""
    parent = [-1] * n_roots + [int(rng.integers(0, i)) for i in range(n_roots, n_nodes)]
    perm = rng.permutation(n_nodes)
    new = {old: int(nw) for old, nw in enumerate(perm)}
    out = [-1] * n_nodes
    for old, p in enumerate(parent):
        out[new[old]] = -1 if p == -1 else new[p]
    has_child = {p for p in out if p != -1}
    leaves = [x for x in range(n_nodes) if x not in has_child]
    return out, leaves


# (the last two: tables of about 14k nodes, as in a paper-shaped rollout batch)
@pytest.mark.parametrize("seed,n_roots,n_nodes", [(0, 1, 30), (1, 4, 200), (2, 64, 3000), (3, 512, 40000),
                                                  (4, 16, 14336), (5, 16, 14337)])
def test_advantage_random_forests(seed, n_roots, n_nodes):
    rng = np.random.default_rng(seed)
    parent, leaves = random_forest(rng, n_roots, n_nodes)
    rewards = rng.choice([0.0, 1.0, 0.5, -1.25], len(leaves)).tolist()
    check_advantage(parent, leaves, rewards)


def test_advantage_of_a_rollout():
    op = R.RolloutParams(prompt_tokens=[100] * 32, width=16, max_depth=8, seg_tokens=64, init_branches=0,
                         p_eos=1 / 200, p_boxed=0.12, p_fail=0.05, p_correct=0.6, seed=4)
    res = R.rollout(op)
    n = max(res.parent) + 1
    parent = [res.parent[x] for x in range(n)]
    leaves = [o.node for _, o in res.outputs]
    rewards = [float(o.reward) for _, o in res.outputs]
    check_advantage(parent, leaves, rewards)


def test_advantage_malformed_table_is_flagged_not_hung():
    parent = [-1, 0, 3, 2, 1]               # 2 <-> 3 is a cycle
    adv, stats = run_advantage(parent, [4, 2], [1.0, 0.0])
    assert stats[3] == 1 and adv[1] == 0
    adv, stats = run_advantage([-1, 0], [5], [1.0])   # leaf id out of range
    assert stats[3] == 1 and adv[0] == 0
