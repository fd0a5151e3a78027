"""Host logic of libtreepo on the CPU (no GPU needed).

The library is loaded and driven through its C ABI on metadata-only trees
(no pool arena: appends move no bytes). The tree operations, the paged block
pool and the tree-walk scheduler are checked bit-exactly against the
oracle's plain tree model and by brute-force enumeration.
"""
import collections
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import oracle
import paper_2508_17445_gb300 as tp
import workloads
from conftest import ROOT, golden

BT = 32


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2508_17445_gb300 import build
    build.build()


def meta_forest(heads=workloads.Heads(8, 2, 64), pool_blocks=1 << 16):
    return tp.Forest(heads.num_q_heads, heads.num_kv_heads, heads.head_dim, pool_blocks, device=None)


# --------------------------------------------------------------------------
# the C ABI
# --------------------------------------------------------------------------
def _declared_functions():
    src = open(os.path.join(ROOT, "include", "treepo.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tp_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    declared = _declared_functions()
    assert len(declared) >= 15
    assert sorted(tp.EXPORTED_SYMBOLS) == declared
    lib = tp.load_library()
    for name in declared:
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", tp.library_path()], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (tp_\w+)", out))
    assert set(declared) <= exported


def test_config_validation():
    bad = [dict(num_q_heads=6, num_kv_heads=4), dict(head_dim=96), dict(block_tokens=16),
           dict(pool_blocks=0), dict(pool_blocks=(1 << 24) + 1), dict(num_kv_heads=0)]
    for kw in bad:
        cfg = dict(num_q_heads=8, num_kv_heads=2, head_dim=64, block_tokens=32, pool_blocks=16)
        cfg.update(kw)
        c = tp.TpConfig(cfg["num_q_heads"], cfg["num_kv_heads"], cfg["head_dim"], cfg["block_tokens"],
                        cfg["pool_blocks"], None, None)
        with pytest.raises(tp.TreepoError) as e:
            tp.tp_tree_create(c)
        assert e.value.code == "INVALID_ARG"
        assert tp.tp_last_error(None)
    c = tp.TpConfig(8, 2, 128, 32, 10, None, None)
    assert tp.tp_pool_bytes(c) == 10 * 2 * 2 * 32 * 128 * 2


# --------------------------------------------------------------------------
# tree operations and the pool, against the oracle model
# --------------------------------------------------------------------------
def _scaled_golden_ops(scale):
    """The hand-worked allocation example with every token count x scale."""
    g = golden("block_allocation.json")
    ops = []
    for step in g["steps"]:
        if "op" in step:
            op = list(step["op"])
            if op[0] == "append":
                op[3] *= scale
            ops.append(("op", op))
        elif "expect_error" in step:
            op = list(step["expect_error"])
            if op[0] == "append":
                op[3] *= scale
            ops.append(("err", op, step["code"]))
        elif "check_path" in step:
            ops.append(("check", step["check_path"][0]))
    return ops, g["pool_blocks"]


def test_golden_allocation_example_scaled_to_32_token_blocks():
    # With every count x16, 2-token blocks become 32-token blocks: the same
    # blocks are handed out, so slot s of the BT=2 example maps to block
    # s // 2. The ABI must agree with the oracle model step by step.
    steps, pool_blocks = _scaled_golden_ops(16)
    f = meta_forest(pool_blocks=pool_blocks)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=pool_blocks)
    ids = {}

    def run(op, model_only=False):
        if op[0] == "root":
            m.add_root(op[1])
            ids[op[1]] = f.add_root()
        elif op[0] == "append":
            m.append(op[1], op[2], op[3])
            tp.tp_append_segment(f.handle, ids[op[1]], op[3])
        elif op[0] == "fork":
            m.fork(op[1], op[2])
            for sid, nid in zip(op[2], f.fork(ids[op[1]], len(op[2]))):
                ids[sid] = nid
        elif op[0] == "prune":
            m.prune(op[1])
            f.prune(ids[op[1]])

    g = golden("block_allocation.json")
    for step in steps:
        if step[0] == "op":
            run(step[1])
        elif step[0] == "err":
            op, code = step[1], step[2]
            with pytest.raises(oracle.OracleError):
                run(op)
            # the model refused; the ABI must refuse with the same code and change nothing
            before = f.stats()
            with pytest.raises(tp.TreepoError) as e:
                if op[0] == "append":
                    tp.tp_append_segment(f.handle, ids.get(op[1], op[1]), op[3])
                elif op[0] == "prune":
                    f.prune(ids[op[1]])
            assert e.value.code == code
            assert f.stats() == before
        else:
            leaf = step[1]
            got = tp.tp_debug_path(f.handle, ids[leaf])
            assert got.tolist() == m.path_slots(leaf).tolist()
    # block-level agreement with the hand-worked BT=2 slots
    for step in g["steps"]:
        if "check_path" in step and step["check_path"][0] == 5:
            blocks_bt2 = sorted({s // 2 for s in step["check_path"][1]})
    assert sorted({s // BT for s in tp.tp_debug_path(f.handle, ids[5]).tolist()}) == blocks_bt2


@pytest.mark.parametrize("seed", range(8))
def test_random_forests_match_oracle_model(seed):
    s = workloads.random_tree(seed=seed, n_prompts=4, max_depth=5, p_prune=0.3, prompt_range=(1, 200),
                              seg_range=(1, 120))
    f = meta_forest(pool_blocks=4096)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=4096).replay(s)
    for sid, nid in ids.items():
        info = f.node_info(nid)
        node = m.nodes[sid]
        assert info["state"] == {"leaf": 0, "frozen": 1, "dead": 2}[node.state]
        if node.state != "dead":
            assert info["n_tokens"] == node.n_tokens
            assert info["n_live_children"] == node.kids_live
    for lf in set(s.leaves):
        assert tp.tp_debug_path(f.handle, ids[lf]).tolist() == m.path_slots(lf).tolist()
    st = f.stats()
    assert st["pool_blocks"] - st["free_blocks"] == m.live_blocks()
    assert st["live_nodes"] == sum(1 for n in m.nodes.values() if n.state != "dead")


def test_full_size_random_divergence_pool_matches_model():
    # config 3 at full size: ~2000 nodes, ~100k blocks, prunes reuse blocks
    s = workloads.random_divergence(seed=0)
    pool_blocks = 1 << 18
    f = meta_forest(heads=s.heads, pool_blocks=pool_blocks)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=pool_blocks).replay(s)
    for lf in s.leaves[::37]:
        assert np.array_equal(tp.tp_debug_path(f.handle, ids[lf]), m.path_slots(lf))
    st = f.stats()
    assert st["pool_blocks"] - st["free_blocks"] == m.live_blocks()


def test_error_codes():
    f = meta_forest(pool_blocks=4)
    r = f.add_root()
    tp.tp_append_segment(f.handle, r, 40)
    with pytest.raises(tp.TreepoError) as e:
        f.fork(r, 0)
    assert e.value.code == "INVALID_ARG"
    a, b = f.fork(r, 2)
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_append_segment(f.handle, r, 1)
    assert e.value.code == "FROZEN"
    with pytest.raises(tp.TreepoError) as e:
        f.prune(r)
    assert e.value.code == "NOT_LEAF"
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_append_segment(f.handle, a, 3 * 32 + 1)   # needs 4 blocks, 2 free
    assert e.value.code == "OOM"
    assert f.node_info(a)["n_tokens"] == 0 and f.stats()["free_blocks"] == 2
    tp.tp_append_segment(f.handle, a, 64)
    f.prune(a)
    with pytest.raises(tp.TreepoError) as e:
        f.prune(a)
    assert e.value.code == "BAD_NODE"
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_schedule(f.handle, [a])
    assert e.value.code == "BAD_NODE"
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_schedule(f.handle, [r])
    assert e.value.code == "NOT_LEAF"
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_get_node_info(f.handle, 999)
    assert e.value.code == "BAD_NODE"
    # an empty leaf under an empty root has no token on its path
    r2 = f.add_root()
    (c,) = f.fork(r2, 1)
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_schedule(f.handle, [c])
    assert e.value.code == "EMPTY_PATH"
    # metadata-only trees refuse device work and device pointers
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_append_segment(f.handle, b, 1, K=_FakePtr(), V=_FakePtr())
    assert e.value.code == "INVALID_ARG"
    # pruning the last leaf frees the whole tree
    f.prune(b)
    assert f.node_info(r)["state"] == 2
    assert f.stats()["free_blocks"] == 4


class _FakePtr:
    def data_ptr(self):
        return 0x1000


def test_wait_probe_needs_a_device_tree():
    f = meta_forest(pool_blocks=4)
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_wait_probe(f.handle, 1_000_000)
    assert e.value.code == "INVALID_ARG"


def test_host_buffer_calls_check_their_arguments():
    import torch
    f = meta_forest(pool_blocks=8)
    r = f.add_root()
    tp.tp_append_segment(f.handle, r, 40)
    q = torch.zeros(1, f.cfg.num_q_heads, f.cfg.head_dim, dtype=torch.bfloat16)
    o, lse = torch.empty_like(q), torch.empty(1, f.cfg.num_q_heads)
    for call in (lambda: tp.tp_decode_host(f.handle, [r], q, o, lse),
                 lambda: tp.tp_prefill_host(f.handle, [r], [1], q, o, lse)):
        with pytest.raises(tp.TreepoError) as e:   # metadata-only trees run no attention
            call()
        assert e.value.code == "INVALID_ARG"
    lib = tp.load_library()
    nodes = np.array([r], dtype=np.int32)
    assert lib.tp_decode_host(f.handle, nodes.ctypes.data, 0, None, None, None, 0) == 0   # n = 0: nothing to do
    assert lib.tp_decode_host(f.handle, nodes.ctypes.data, -1, None, None, None, 0) == -1
    with pytest.raises(ValueError):   # the binding takes contiguous CPU tensors only
        tp.tp_decode_host(f.handle, [r], q.transpose(1, 2), o, lse)


def test_fork_of_frozen_node_adds_children():
    f = meta_forest()
    r = f.add_root()
    tp.tp_append_segment(f.handle, r, 5)
    a = f.fork(r, 1)
    b = f.fork(r, 2)
    assert f.node_info(r)["n_live_children"] == 3
    assert len(set(a + b)) == 3
    for c in a + b:
        assert f.node_info(c)["path_tokens"] == 5


# --------------------------------------------------------------------------
# scheduler: bit-exact coverage by enumeration
# --------------------------------------------------------------------------
def _expand(tiles):
    out = []
    for w in tiles:
        blk, valid = int(w) >> 7, (int(w) & 127) + 1
        out += [blk * BT + r for r in range(valid)]
    return out


def check_merge_records(S):
    """Each occurrence's fixed-size merge record holds its CSR slots: count,
    then the slots in order, zero-padded; -1 when it has more than 15."""
    rec = S["merge_rec"]
    assert rec.shape == (len(S["merge_off"]) - 1, 16)
    for i in range(rec.shape[0]):
        beg, end = int(S["merge_off"][i]), int(S["merge_off"][i + 1])
        if end - beg >= 16:
            assert rec[i, 0] == -1 and not rec[i, 1:].any()
        else:
            assert rec[i, 0] == end - beg
            assert rec[i, 1:1 + end - beg].tolist() == S["merge_slot"][beg:end].tolist()
            assert not rec[i, 1 + end - beg:].any()


def check_schedule(f, ids, model, script, leaves_sid, flags=0):
    heads = script.heads
    g = heads.group
    leaves = [ids[x] for x in leaves_sid]
    S = tp.tp_debug_schedule(f.handle, leaves, flags)
    assert S["group"] == g
    # a call reading less than 1 MiB of K/V (its path blocks, counted whole:
    # each shared block once, or once per leaf without sharing) keeps every
    # unit on mma.sync unless tcgen05 is forced
    nodes = [x for x in {y for lf in leaves_sid for y in model.path_nodes(lf)}] if not flags & tp.TP_DECODE_NO_SHARE \
        else [y for lf in leaves_sid for y in model.path_nodes(lf)]
    blocks = sum(-(-model.nodes[x].n_tokens // BT) for x in nodes)
    small = blocks * heads.num_kv_heads * BT * heads.head_dim * 4 < (1 << 20) and not flags & tp.TP_DECODE_ALL_TCGEN05
    all_tc = not flags & tp.TP_MMA_SYNC and not small and not (
        flags & tp.TP_DECODE_TCGEN05 and not flags & tp.TP_DECODE_ALL_TCGEN05)
    if small:
        assert S["n_tc_units"] == 0
    covered = collections.defaultdict(list)
    slots_of = collections.defaultdict(set)
    chunk_reads = collections.Counter()
    for u in S["units"]:
        toff, nt, ooff, row0, nrows, sbase, kvh, kind = (int(x) for x in u)
        assert 0 <= kvh < heads.num_kv_heads
        if kind == 0:                      # CUDA-core: one leaf group, < 16 rows
            assert nrows < 16 and flags & tp.TP_DECODE_CUDA_CORE_SMALL
        elif kind == 1:                    # mma.sync: one 16-row tile (all-tcgen05), else 64-row blocks
            if all_tc:
                assert row0 == 0 and 1 <= nrows <= 16
            else:
                assert 1 <= nrows <= 64
            if flags & tp.TP_DECODE_CUDA_CORE_SMALL:
                assert nrows >= 16 or row0 > 0
        else:                              # tcgen05: stacked rows in 128-row blocks
            assert kind == 2 and not flags & tp.TP_MMA_SYNC and not small
            assert 1 <= nrows <= 128
            if all_tc:
                assert row0 > 0 or nrows >= 17
            else:
                assert nt >= 32 and (row0 > 0 or nrows >= 64)
        tok = _expand(S["tiles"][toff:toff + nt])
        assert len(tok) > 0
        if row0 == 0:
            chunk_reads[(toff, kvh)] += 1
        for r in range(nrows):
            item_row = row0 + r
            p, j = divmod(item_row, g)
            i = int(S["occ"][ooff + p])
            qh = kvh * g + j
            covered[(i, qh)] += tok
            slots_of[(i, qh)].add(sbase + p)
    n = len(leaves)
    check_merge_records(S)
    for i in range(n):
        want = sorted(model.path_slots(leaves_sid[i]).tolist())
        mslots = S["merge_slot"][S["merge_off"][i]:S["merge_off"][i + 1]].tolist()
        assert len(mslots) == len(set(mslots))
        for qh in range(heads.num_q_heads):
            assert sorted(covered[(i, qh)]) == want, (i, qh)
            assert set(mslots) == slots_of[(i, qh)]
    assert all(c == 1 for c in chunk_reads.values())
    return S


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("flags", [0, tp.TP_DECODE_NO_SHARE, tp.TP_DECODE_CUDA_CORE_SMALL, tp.TP_DECODE_TCGEN05,
                                   tp.TP_DECODE_ALL_TCGEN05, tp.TP_MMA_SYNC])
def test_schedule_covers_every_path_token_once(seed, flags):
    s = workloads.random_tree(seed=seed, n_prompts=3, max_depth=5, prompt_range=(1, 300), seg_range=(1, 150),
                              heads=workloads.Heads(8, 2, 64))
    f = meta_forest(heads=s.heads, pool_blocks=1 << 14)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=1 << 14).replay(s)
    check_schedule(f, ids, m, s, s.leaves, flags)


@pytest.mark.parametrize("name,kw", [("tiny", {}), ("qwen7b", {"n_prompts": 2}),
                                     ("random_divergence", {"n_prompts": 2, "depth": 6}),
                                     ("wide_prefix", {"n_prompts": 1}), ("no_sharing", {"n_seqs": 4})])
def test_schedule_on_named_workloads(name, kw):
    s = workloads.by_name(name, **kw)
    f = meta_forest(heads=s.heads, pool_blocks=1 << 16)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=1 << 16).replay(s)
    S = check_schedule(f, ids, m, s, s.leaves)
    # sharing: tiles read (per kv head) == unique blocks on the union of paths
    uniq_blocks = set()
    for lf in s.leaves:
        uniq_blocks |= {x // BT for x in m.path_slots(lf).tolist()}
    read = sum(int(u[1]) for u in S["units"] if int(u[3]) == 0)
    assert read == len(uniq_blocks) * s.heads.num_kv_heads


def test_long_shared_node_is_cut_into_chunks():
    s = workloads.shared_prompt()
    f = meta_forest(heads=s.heads, pool_blocks=1 << 10)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=1 << 10).replay(s)
    S = check_schedule(f, ids, m, s, s.leaves)
    # 63 prompt blocks, 24 rows per kv head: chunks of >= 30 blocks
    prompt_units = [u for u in S["units"] if int(u[1]) > 10]
    assert len({int(u[0]) for u in prompt_units}) >= 2
    assert all(int(u[1]) >= 30 for u in prompt_units)


def test_schedule_without_sharing_reads_every_path():
    s = workloads.wide_prefix(n_prompts=1)
    f = meta_forest(heads=s.heads, pool_blocks=1 << 16)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT, pool_blocks=1 << 16).replay(s)
    S = check_schedule(f, ids, m, s, s.leaves, tp.TP_DECODE_NO_SHARE)
    read = sum(int(u[1]) for u in S["units"])
    assert read == len(s.leaves) * (3328 // BT) * s.heads.num_kv_heads


def test_duplicate_leaves_and_empty_set():
    s = workloads.tiny()
    f = meta_forest(heads=s.heads)
    ids = f.replay(s.ops)
    m = oracle.OracleForest(block_tokens=BT).replay(s)
    leaves = [s.leaves[0], s.leaves[3], s.leaves[0], s.leaves[0]]
    check_schedule(f, ids, m, s, leaves)
    S = tp.tp_debug_schedule(f.handle, [])
    assert len(S["units"]) == 0 and len(S["merge_off"]) == 1
