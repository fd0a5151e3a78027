"""Host side of the tree sampler (no GPU): the library's Algorithm 1 driver
on a metadata-only tree against the oracle's, event for event; the branch
split against the oracle's; the decode-loop token append's bookkeeping."""
import numpy as np
import pytest

import oracle.rollout as R
import paper_2508_17445_gb300 as tp


def product_params(op: R.RolloutParams, **extra):
    kw = dict(width=op.width, max_depth=op.max_depth, seg_tokens=op.seg_tokens, arity=op.arity,
              init_branches=op.init_branches, policy=op.policy, fallback=int(op.fallback),
              temperature=op.temperature, p_eos=op.p_eos, p_boxed=op.p_boxed, p_fail=op.p_fail,
              p_correct=op.p_correct, seed=op.seed)
    kw.update(extra)
    return tp.rollout_params(list(op.prompt_tokens), **kw)


def random_params(seed: int) -> R.RolloutParams:
    rng = np.random.default_rng(500 + seed)
    return R.RolloutParams(
        prompt_tokens=[int(x) for x in rng.integers(1, 100, int(rng.integers(1, 6)))],
        width=int(rng.integers(1, 20)), max_depth=int(rng.integers(1, 8)), seg_tokens=int(rng.integers(1, 40)),
        arity=int(rng.integers(1, 4)), init_branches=int(rng.integers(0, 5)), policy=int(rng.integers(0, 3)),
        fallback=bool(rng.integers(0, 2)), temperature=float(rng.uniform(0.2, 5)),
        p_eos=float(rng.choice([0.0, 0.01, 0.1, 0.5])), p_boxed=float(rng.uniform(0, 0.6)),
        p_fail=float(rng.uniform(0, 0.5)), p_correct=float(rng.uniform(0, 1)), seed=int(rng.integers(0, 2**63)))


@pytest.mark.parametrize("seed", range(24))
def test_dry_rollout_matches_oracle_event_for_event(seed):
    op = random_params(seed)
    res = R.rollout(op)
    f = tp.Forest(8, 2, 64, pool_blocks=1 << 16, device=None)
    ev, st = f.rollout(product_params(op))
    np.testing.assert_array_equal(ev, R.events_array(res))
    kinds = ev[:, 0]
    assert st["segments"] == int((kinds == R.EV_SEGMENT).sum())
    assert st["outputs"] == int((kinds == R.EV_OUTPUT).sum())
    assert st["fallbacks"] == int((kinds == R.EV_FALLBACK).sum())
    assert st["tokens"] == int(ev[kinds == R.EV_SEGMENT, 4].sum())
    assert st["nodes"] == len(res.parent) and st["decode_calls"] == 0
    s = f.stats()
    assert s["live_nodes"] == 0 and s["free_blocks"] == s["pool_blocks"]   # every trajectory released
    for x, par in res.parent.items():                                       # same tree
        assert f.node_info(x)["parent"] == par


def test_paper_shaped_rollout_matches_oracle():
    # 14 x 512 segments, w = 16, binary budget, prompts up to 1024 tokens
    op = R.RolloutParams(prompt_tokens=[1024, 640, 300, 877], width=16, max_depth=14, seg_tokens=512,
                         init_branches=2, p_eos=1 / 2048, p_boxed=0.04, p_fail=0.03, seed=11)
    f = tp.Forest(28, 4, 128, pool_blocks=1 << 20, device=None)
    ev, st = f.rollout(product_params(op))
    np.testing.assert_array_equal(ev, R.events_array(R.rollout(op)))
    assert st["outputs"] <= 64 and st["peak_blocks"] > 0


def test_rollout_on_a_nonempty_tree_continues_the_ids():
    f = tp.Forest(8, 2, 64, pool_blocks=1 << 14, device=None)
    r = f.add_root()
    tp.tp_append_segment(f.handle, r, 40, None, None)
    f.fork(r, 3)
    op = random_params(3)
    ev, _ = f.rollout(product_params(op))
    np.testing.assert_array_equal(ev, R.events_array(R.rollout(op, first_node=4)))
    assert f.stats()["live_nodes"] == 4           # the earlier tree is untouched


@pytest.mark.parametrize("policy", [R.BRANCH_LOGP_HIGH, R.BRANCH_LOGP_LOW])
def test_logprob_policies_change_the_tree(policy):
    base = random_params(7)
    base.policy, base.p_fail, base.p_boxed, base.p_eos = R.BRANCH_EVEN, 0.1, 0.05, 0.0
    base.width, base.max_depth, base.arity = 16, 6, 2
    other = R.RolloutParams(**{**base.__dict__, "policy": policy})
    f = tp.Forest(8, 2, 64, pool_blocks=1 << 16, device=None)
    ev_even, _ = f.rollout(product_params(base))
    ev_lp, _ = f.rollout(product_params(other))
    assert not np.array_equal(ev_even[:, 3:5], ev_lp[:, 3:5])


def test_branch_assign_matches_oracle():
    rng = np.random.default_rng(4)
    for _ in range(400):
        n = int(rng.integers(1, 40))
        budget = n + int(rng.integers(0, 200))
        policy = int(rng.integers(0, 3))
        lp = rng.normal(-1.0, float(rng.uniform(0.01, 3)), n)
        if rng.random() < 0.2:
            lp[: n // 2] = lp[0]                                        # ties
        T = float(rng.choice([0.1, 1.0, 2.0, 5.0, 1e6]))
        want = R.branch_split(list(lp), n, budget, policy, T)
        assert tp.tp_branch_assign(lp, n, budget, policy, T) == want


def test_branch_assign_rejects_bad_arguments():
    for args in (([0.0, 0.0], 2, 1, 0, 1.0), ([0.0], 1, 3, 1, 0.0), ([np.nan], 1, 3, 1, 1.0),
                 ([0.0], 1, 3, 9, 1.0)):
        with pytest.raises(tp.TreepoError):
            tp.tp_branch_assign(*args)
    assert tp.tp_branch_assign(None, 0, 0, 0) == []


def test_rollout_parameter_validation():
    f = tp.Forest(8, 2, 64, pool_blocks=1 << 10, device=None)
    good = dict(width=4, max_depth=2, seg_tokens=8)
    for bad in (dict(width=0), dict(max_depth=0), dict(seg_tokens=0), dict(arity=0), dict(init_branches=-1),
                dict(policy=5), dict(policy=1, temperature=0.0), dict(decode=1)):
        with pytest.raises(tp.TreepoError) as e:
            f.rollout(tp.rollout_params([5], **{**good, **bad}))
        assert e.value.code == "INVALID_ARG"
    with pytest.raises(tp.TreepoError):
        f.rollout(tp.rollout_params([0], **good))
    # a pool too small for the prompts: OOM, reported
    small = tp.Forest(8, 2, 64, pool_blocks=2, device=None)
    with pytest.raises(tp.TreepoError) as e:
        small.rollout(tp.rollout_params([100], **good))
    assert e.value.code == "OOM"


def test_event_capacity_is_checked():
    f = tp.Forest(8, 2, 64, pool_blocks=1 << 12, device=None)
    with pytest.raises(tp.TreepoError):
        f.rollout(tp.rollout_params([5, 5], width=4, max_depth=3, seg_tokens=4), cap_events=3)


# ------------------------------------------------------ decode-loop append --
def test_append_tokens_equals_one_token_appends():
    rng = np.random.default_rng(9)
    a = tp.Forest(8, 2, 64, pool_blocks=4096, device=None)
    b = tp.Forest(8, 2, 64, pool_blocks=4096, device=None)
    leaves_a, leaves_b = [], []
    for forest, leaves in ((a, leaves_a), (b, leaves_b)):
        for _ in range(3):
            r = forest.add_root()
            tp.tp_append_segment(forest.handle, r, 45, None, None)
            leaves.extend(forest.fork(r, 3))
    for step in range(70):
        pick = sorted(rng.choice(len(leaves_a), size=int(rng.integers(1, len(leaves_a) + 1)), replace=False))
        a.append_tokens([leaves_a[i] for i in pick])
        for i in pick:
            tp.tp_append_segment(b.handle, leaves_b[i], 1, None, None)
        if step % 17 == 5:                      # interleave prunes
            a.prune(leaves_a[-1]), b.prune(leaves_b[-1])
            leaves_a.pop(), leaves_b.pop()
    for x, y in zip(leaves_a, leaves_b):
        np.testing.assert_array_equal(tp.tp_debug_path(a.handle, x), tp.tp_debug_path(b.handle, y))
    assert a.stats() == b.stats()


def test_append_tokens_errors_leave_the_tree_unchanged():
    f = tp.Forest(8, 2, 64, pool_blocks=3, device=None)
    r = f.add_root()
    tp.tp_append_segment(f.handle, r, 32, None, None)
    k1, k2 = f.fork(r, 2)
    before = f.stats()
    for nodes, code in (([k1, k1], "INVALID_ARG"), ([r], "FROZEN"), ([999], "BAD_NODE")):
        with pytest.raises(tp.TreepoError) as e:
            f.append_tokens(nodes)
        assert e.value.code == code
    assert f.stats() == before
    tp.tp_append_segment(f.handle, k1, 1, None, None)      # k1 takes the 2nd block
    f.append_tokens([k2, k1])                              # k2 takes the 3rd, k1 stays in its block
    tp.tp_append_segment(f.handle, k1, 30, None, None)     # k1's block is now full
    before = f.stats()
    with pytest.raises(tp.TreepoError) as e:               # k1 needs a 4th block
        f.append_tokens([k2, k1])
    assert e.value.code == "OOM"
    assert f.stats() == before
    assert f.node_info(k1)["n_tokens"] == 32 and f.node_info(k2)["n_tokens"] == 1
    f.append_tokens([k2])
    assert f.node_info(k2)["n_tokens"] == 2
    assert f.append_tokens([]) is None
