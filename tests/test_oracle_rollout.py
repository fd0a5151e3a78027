"""Pins for the sampler and advantage oracles (oracle/rollout.py,
oracle/advantage.py): published generator outputs, hand-computed values,
closed-form tree shapes and invariants -- nothing taken from the oracle
itself. Each is chosen so that a plausible slip (an off-by-one stream index,
a budget computed at the wrong depth, a fallback taken while paths remain,
a sub-group that includes the leaf itself, a std over the wrong set) fails.
"""
import math
from collections import Counter, defaultdict

import numpy as np
import pytest

import oracle.advantage as A
import oracle.rollout as R
from conftest import golden


# ------------------------------------------------------------- generator --
def test_splitmix64_published_outputs():
    for seq in golden("splitmix64.json")["sequences"]:
        want = [int(x, 0) for x in seq["outputs"]]
        assert [R.splitmix64(seq["seed"], i) for i in range(len(want))] == want


def test_uniform_is_top_53_bits_and_covers_unit_interval():
    seed = 99
    xs = np.array([R.uniform(seed, R.TAG_EOS, 5, t) for t in range(20000)])
    assert xs.min() >= 0.0 and xs.max() < 1.0
    assert abs(xs.mean() - 0.5) < 0.01 and abs(xs.var() - 1 / 12) < 0.005
    x = R.uniform(seed, 4, 5, 6, 7)
    assert x == (R.splitmix64(seed, (4 << 60) | (5 << 32) | (6 << 12) | 7) >> 11) / 2.0 ** 53


def test_counter_fields_do_not_alias():
    seen = {R.counter(t, a, b, c) for t in (1, 7) for a in (0, 1, (1 << 28) - 1) for b in (0, 1, (1 << 20) - 1)
            for c in (0, 1, 4095)}
    assert len(seen) == 2 * 3 * 3 * 3


def test_synth_rows_bit_layout():
    bits = R.synth_rows(5, R.TAG_K, [3, 3, 9], [0, 1, 0], 2, 8)
    assert bits.shape == (3, 2, 8) and bits.dtype == np.uint16
    vals = np.abs(R.bf16_to_f64(bits))
    assert vals.min() >= 0.125 and vals.max() < 2.0
    # word 1 of row (node 3, token 1) holds elements 4..7, low 16 bits first
    h = R.splitmix64(5, R.counter(R.TAG_K, 3, 1, 1))
    for lane in range(4):
        r = (h >> (16 * lane)) & 0xFFFF
        sign, expo, mant = r >> 15, 124 + ((r >> 7) & 3), r & 0x7F
        assert R.bf16_to_f64(bits[1:2, 0, 4 + lane])[0] == (-1) ** sign * 2.0 ** (expo - 127) * (1 + mant / 128)
    big = R.bf16_to_f64(R.synth_rows(1, R.TAG_V, list(range(64)), [7] * 64, 4, 64))
    assert abs((big > 0).mean() - 0.5) < 0.03
    # unit-normal scale: E[x^2] = E[(1 + m)^2] * mean(4^e), e in -3..0, m uniform on [0, 1)
    want_ms = (7 / 3) * (4.0 ** -3 + 4.0 ** -2 + 4.0 ** -1 + 1) / 4
    assert abs((big ** 2).mean() - want_ms) < 0.05 * want_ms


# ---------------------------------------------------------- branch split --
def test_branch_split_hand_values():
    assert R.branch_split(None, 3, 10, R.BRANCH_EVEN) == [4, 3, 3]
    assert R.branch_split(None, 4, 4, R.BRANCH_EVEN) == [1, 1, 1, 1]
    # softmax([2, 0]) = (0.8808, 0.1192); 10 extra -> quotas 8.808, 1.192
    assert R.branch_split([2.0, 0.0], 2, 12, R.BRANCH_LOGP_HIGH, 1.0) == [10, 2]
    assert R.branch_split([2.0, 0.0], 2, 12, R.BRANCH_LOGP_LOW, 1.0) == [2, 10]
    # T = 2 halves the logits: softmax([1, 0]) = (0.7311, 0.2689); 6 extra
    assert R.branch_split([2.0, 0.0], 2, 8, R.BRANCH_LOGP_HIGH, 2.0) == [5, 3]


def test_branch_split_properties():
    rng = np.random.default_rng(0)
    for _ in range(300):
        n = int(rng.integers(1, 12))
        budget = n + int(rng.integers(0, 40))
        lp = list(rng.normal(-1.0, 0.7, n))
        T = float(rng.uniform(0.2, 5.0))
        hi = R.branch_split(lp, n, budget, R.BRANCH_LOGP_HIGH, T)
        lo = R.branch_split(lp, n, budget, R.BRANCH_LOGP_LOW, T)
        for split in (hi, lo):
            assert sum(split) == budget and min(split) >= 1
        assert lo == R.branch_split([-x for x in lp], n, budget, R.BRANCH_LOGP_HIGH, T)
        order = np.argsort(lp)
        assert all(hi[order[k]] <= hi[order[k + 1]] + 1 for k in range(n - 1))   # monotone up to rounding
        # equal log-probabilities (or T -> infinity) give the even split
        assert R.branch_split([0.3] * n, n, budget, R.BRANCH_LOGP_HIGH, T) == R.branch_split(None, n, budget, 0)
        # (which paths get the leftover units then rests on tiny differences)
        assert sorted(R.branch_split(lp, n, budget, R.BRANCH_LOGP_HIGH, 1e12)) == \
            sorted(R.branch_split(None, n, budget, 0))


def test_branch_split_rejects_bad_arguments():
    with pytest.raises(ValueError):
        R.branch_split(None, 3, 2, R.BRANCH_EVEN)
    with pytest.raises(ValueError):
        R.branch_split([0.0], 1, 3, R.BRANCH_LOGP_HIGH, 0.0)


# --------------------------------------------------------------- sampler --
def _by_kind(res):
    out = defaultdict(list)
    for e in res.events:
        out[e[0]].append(e)
    return out


def test_full_binary_tree_closed_form():
    # no early stop: 2, 4, 8, 16, 16, 16 paths generate segments 1..6
    p = R.RolloutParams(prompt_tokens=[50, 70], width=16, max_depth=6, seg_tokens=8, arity=2, init_branches=2)
    res = R.rollout(p)
    ev = _by_kind(res)
    assert len(ev[R.EV_SEGMENT]) == 2 * (2 + 4 + 8 + 16 + 16 + 16)
    per_depth = Counter((e[1], e[3]) for e in ev[R.EV_SEGMENT])
    assert [per_depth[(0, d)] for d in range(1, 7)] == [2, 4, 8, 16, 16, 16]
    assert all(e[4] == 8 and e[5] == (R.SEG_MAX_DEPTH if e[3] == 6 else 0) for e in ev[R.EV_SEGMENT])
    assert len(ev[R.EV_FORK]) == 2 * (1 + 2 + 4 + 8 + 16 + 16)
    outs = ev[R.EV_OUTPUT]
    assert len(outs) == 32 and all(e[3] == 6 and e[4] == 0 for e in outs)
    assert len(ev[R.EV_PRUNE]) == 32 and not ev[R.EV_FALLBACK]
    assert [e[3] for e in ev[R.EV_DONE]] == [16, 16]
    assert len(res.parent) == 2 * (1 + 62)


def test_ternary_budget_capped_by_width():
    # b0 = 1, N = 3, w = 10: budgets 1, 3, 9, then 10 (9 paths -> one forks twice)
    p = R.RolloutParams(prompt_tokens=[5], width=10, max_depth=4, seg_tokens=4, arity=3, init_branches=1)
    ev = _by_kind(R.rollout(p))
    assert Counter(e[3] for e in ev[R.EV_SEGMENT]) == {1: 1, 2: 3, 3: 9, 4: 10}
    last_forks = [e[4] for e in ev[R.EV_FORK]][-9:]
    assert last_forks == [2] + [1] * 8


def test_all_segments_fail():
    p = R.RolloutParams(prompt_tokens=[9, 9, 9], width=16, max_depth=5, seg_tokens=4, init_branches=3, p_fail=1.0)
    ev = _by_kind(R.rollout(p))
    assert len(ev[R.EV_OUTPUT]) == 9 and all(e[3] == 1 and e[4] == 0 and e[5] == 0 for e in ev[R.EV_OUTPUT])
    assert not ev[R.EV_FALLBACK] and [e[3] for e in ev[R.EV_DONE]] == [3, 3, 3]


def test_all_boxed_refills_width_by_fallback():
    # every segment answers at depth 1: b0 outputs, then one fallback path
    # from the root (the only boundary of a one-segment trajectory) per pass
    w, b0 = 7, 2
    p = R.RolloutParams(prompt_tokens=[12, 20], width=w, max_depth=5, seg_tokens=4, init_branches=b0,
                        p_boxed=1.0, p_correct=1.0)
    res = R.rollout(p)
    ev = _by_kind(res)
    assert len(ev[R.EV_FALLBACK]) == 2 * (w - b0)
    assert all(e[4] == 0 and e[3] == res.path(e[2])[0] for e in ev[R.EV_FALLBACK])
    assert len(ev[R.EV_OUTPUT]) == 2 * w and all(e[4] == 1 and e[5] == 1 for e in ev[R.EV_OUTPUT])
    assert [e[3] for e in ev[R.EV_DONE]] == [w, w]


def test_truncated_trajectories_are_not_fallback_candidates():
    # max depth 1 without EOS or a boxed answer: b0 < w outputs, none of
    # them a candidate, so no fallback and every leaf is pruned at once
    p = R.RolloutParams(prompt_tokens=[8, 8], width=16, max_depth=1, seg_tokens=4, init_branches=3)
    ev = _by_kind(R.rollout(p))
    assert len(ev[R.EV_OUTPUT]) == 6 and all(e[4] == 0 for e in ev[R.EV_OUTPUT])
    assert not ev[R.EV_FALLBACK]
    order = [e[0] for e in R.rollout(p).events if e[0] in (R.EV_OUTPUT, R.EV_PRUNE)]
    assert order == [R.EV_OUTPUT, R.EV_PRUNE] * 6


def test_every_token_eos_gives_one_token_segments():
    p = R.RolloutParams(prompt_tokens=[3], width=4, max_depth=3, seg_tokens=16, p_eos=1.0, fallback=False)
    ev = _by_kind(R.rollout(p))
    assert all(e[4] == 1 and e[5] & R.SEG_EOS for e in ev[R.EV_SEGMENT])
    assert len(ev[R.EV_OUTPUT]) == 2         # both initial paths end at depth 1; no fallback


def _check_invariants(p, res):
    alive, live_kids, outputs, active = set(), Counter(), Counter(), defaultdict(set)
    q_done, cands = set(), set()
    seg_of = {}
    for e in res.events:
        kind, q, node = e[0], e[1], e[2]
        if kind == R.EV_ROOT:
            alive.add(node)
            assert p.init_branches == 0 or e[4] == p.init_branches
            assert 2 <= e[4] <= 8 if p.init_branches == 0 else True
        elif kind == R.EV_FORK:
            assert node in alive and q not in q_done
            kids = list(range(e[3], e[3] + e[4]))
            assert all(res.parent[c] == node and res.depth[c] == res.depth[node] + 1 for c in kids)
            alive.update(kids)
            live_kids[node] += e[4]
            active[q].update(kids)
            active[q].discard(node)
            assert len(active[q]) + outputs[q] <= p.width
        elif kind == R.EV_SEGMENT:
            assert node in active[q] and 1 <= e[4] <= p.seg_tokens and 1 <= e[3] <= p.max_depth
            assert bool(e[5] & R.SEG_MAX_DEPTH) == (e[3] == p.max_depth)
            assert bool(e[5] & R.SEG_EOS) == (e[4] < p.seg_tokens or
                                              (p.p_eos > 0 and R.uniform(p.seed, R.TAG_EOS, node, e[4] - 1) < p.p_eos))
            seg_of[node] = e
        elif kind == R.EV_OUTPUT:
            outputs[q] += 1
            if e[4]:
                cands.add(node)
            active[q].discard(node)
            assert outputs[q] <= p.width
            s = seg_of[node]
            assert e[4] == int(bool(s[5] & (R.SEG_EOS | R.SEG_BOXED_BIT)) and not s[5] & R.SEG_FAILED)
        elif kind == R.EV_PRUNE:
            assert node in alive and live_kids[node] == 0
            x = node
            while x != -1 and live_kids[x] == 0:
                alive.discard(x)
                x = res.parent[x]
                if x != -1:
                    live_kids[x] -= 1
        elif kind == R.EV_FALLBACK:
            assert not active[q] and outputs[q] < p.width and node in alive and node in cands
            assert e[3] in res.path(node) and res.depth[e[3]] == e[4] < res.depth[node]
        elif kind == R.EV_DONE:
            assert not active[q] and e[3] == outputs[q]
            q_done.add(q)
    assert not alive and len(q_done) == len(p.prompt_tokens)


@pytest.mark.parametrize("seed", range(16))
def test_rollout_invariants_random_parameters(seed):
    rng = np.random.default_rng(100 + seed)
    p = R.RolloutParams(
        prompt_tokens=[int(x) for x in rng.integers(1, 80, int(rng.integers(1, 5)))],
        width=int(rng.integers(1, 17)), max_depth=int(rng.integers(1, 7)), seg_tokens=int(rng.integers(1, 24)),
        arity=int(rng.integers(1, 4)), init_branches=int(rng.integers(0, 4)), policy=int(rng.integers(0, 3)),
        fallback=bool(rng.integers(0, 2)), temperature=float(rng.uniform(0.3, 4)),
        p_eos=float(rng.choice([0.0, 0.02, 0.2])), p_boxed=float(rng.uniform(0, 0.5)),
        p_fail=float(rng.uniform(0, 0.4)), p_correct=0.5, seed=seed)
    _check_invariants(p, R.rollout(p))


def test_branching_follows_the_depth_budget():
    # with early stops, the paths generating depth j+1 of a query number
    # max(min(b0 N^j, w - outputs), continuing paths)
    p = R.RolloutParams(prompt_tokens=[30, 30, 30], width=12, max_depth=6, seg_tokens=6, arity=2,
                        init_branches=2, p_fail=0.25, p_boxed=0.1, fallback=False, seed=3)
    res = R.rollout(p)
    outputs, segs = Counter(), defaultdict(Counter)
    for e in res.events:
        if e[0] == R.EV_SEGMENT:
            segs[e[1]][e[3]] += 1
    # replay the outputs depth by depth
    out_by = defaultdict(Counter)
    for e in res.events:
        if e[0] == R.EV_OUTPUT:
            out_by[e[1]][e[3]] += 1
    for q in range(3):
        done_before = 0
        for j in range(1, p.max_depth):
            cont = segs[q][j] - out_by[q][j]
            done_before += out_by[q][j]
            if cont == 0:
                break
            want = max(min(2 * 2 ** j, p.width - done_before), cont)
            assert segs[q][j + 1] == want, (q, j)


# -------------------------------------------------------------- advantage --
def test_advantage_hand_example():
    g = golden("tree_advantage_figure.json")
    adv, st = A.tree_advantage(g["parent"], g["leaves"], g["rewards"])
    a = np.array(g["A_times_3"]) / 3
    std = math.sqrt(g["std_squared_times_9"] / 9)
    assert st["accepted"] == 8 and abs(st["mean"]) < 1e-15 and abs(st["std"] - std) < 1e-15
    np.testing.assert_allclose(adv, a / std, rtol=0, atol=1e-14)


def test_advantage_flat_tree_is_grpo_numerator():
    rng = np.random.default_rng(1)
    r = rng.integers(0, 2, 16).astype(float)
    r[0], r[1] = 0, 1
    parent = [-1] + [0] * 16
    adv, st = A.tree_advantage(parent, list(range(1, 17)), r)
    grpo = r - r.mean()
    np.testing.assert_allclose(adv, grpo / grpo.std(), rtol=0, atol=1e-13)


def test_advantage_rejects_uniform_queries_and_is_invariant():
    rng = np.random.default_rng(2)
    # two queries: root 0 (binary depth 2) and root 7 whose rewards all agree
    parent = [-1, 0, 0, 1, 1, 2, 2, -1, 7, 7, 8, 8]
    leaves = [3, 4, 5, 6, 9, 10, 11]
    r = np.array([1.0, 0.0, 0.5, 1.0, 2.0, 2.0, 2.0])
    adv, st = A.tree_advantage(parent, leaves, r)
    assert st["accepted"] == 4 and np.all(adv[4:] == 0)
    one, _ = A.tree_advantage(parent, leaves[:4], r[:4])
    np.testing.assert_allclose(adv[:4], one, atol=1e-14)        # the rejected query is left out of the std
    for shift, scale in ((3.0, 1.0), (0.0, 2.5), (-1.0, 0.1)):
        a2, _ = A.tree_advantage(parent, leaves, r * scale + shift)
        np.testing.assert_allclose(a2, adv, atol=1e-12)
    # relabel the nodes: same advantages
    perm = list(rng.permutation(len(parent)))
    new = {old: new for new, old in enumerate(perm)}
    parent2 = [-1] * len(parent)
    for old, p in enumerate(parent):
        parent2[new[old]] = -1 if p == -1 else new[p]
    a3, _ = A.tree_advantage(parent2, [new[x] for x in leaves], r)
    np.testing.assert_allclose(a3, adv, atol=1e-14)


def test_advantage_leaf_root_and_single_output():
    adv, st = A.tree_advantage([-1, -1, 1, 1], [0, 2, 3], [1.0, 0.0, 1.0])
    assert adv[0] == 0 and st["accepted"] == 2            # a root leaf has no sub-group
    adv, st = A.tree_advantage([-1, 0], [1], [1.0])       # one trajectory: all rewards agree
    assert st["accepted"] == 0 and adv[0] == 0
