"""Prefill schedules (no GPU): every query token reads each token of its
path it may see -- and nothing past its own position -- exactly once, over
its merge slots or through the one unit that writes its output directly,
with rows in whole GQA groups."""
import numpy as np
import pytest

import oracle
import paper_2508_17445_gb300 as tp
import workloads


def metadata_forest(script):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=script.upper_bound_blocks(32) + 8,
                  device=None)
    ids = f.replay(script.ops, kv_fn=None)
    return f, ids


def check_prefill_coverage(f, model, ids, nodes_sid, counts, flags=0):
    g = f.cfg.num_q_heads // f.cfg.num_kv_heads
    hkv = f.cfg.num_kv_heads
    nodes = [ids[x] for x in nodes_sid]
    d = tp.tp_debug_prefill_schedule(f.handle, nodes, counts, flags)
    units, tiles = d["units"], d["tiles"]
    tc = not (flags & tp.TP_MMA_SYNC)
    assert len(d["vis"]) == sum(counts) and np.array_equal(d["occ"], np.arange(sum(counts)))
    assert np.all(units[:, 7] == (2 if tc else 1)) and np.all(units[:, 4] % g == 0)
    assert np.all(units[:, 4] <= (128 if tc else 64))
    valid = (tiles & 127) + 1
    block = tiles >> 7
    # slot -> (occurrence, unit, kv head); units with slot_base < 0 write the
    # final output of their rows directly (the rows' only unit)
    owner, direct = {}, {}
    for ui, u in enumerate(units):
        toff, nt, occ_off, row0, n_rows, slot_base, kvh = (int(x) for x in u[:7])
        assert row0 == 0
        for p in range(n_rows // g):
            if slot_base < 0:
                direct.setdefault(occ_off + p, []).append((occ_off + p, ui, kvh))
            else:
                owner.setdefault(slot_base + p, []).append((occ_off + p, ui, kvh))
    assert "merge_rec" not in d      # prefill rows merge through the CSR
    r = 0
    for x_sid, mq in zip(nodes_sid, counts):
        chain = model.path_nodes(x_sid, True)
        path_slots = [model.nodes[y].blocks[t // 32] * 32 + t % 32
                      for y in chain for t in range(model.nodes[y].n_tokens)]
        P = len(path_slots)
        for j in range(mq):
            q = r + j
            vis = P - mq + j + 1
            assert d["vis"][q] == vis
            seen = []
            slots = d["merge_slot"][d["merge_off"][q]:d["merge_off"][q + 1]]
            assert (len(slots) == 0) == (q in direct)
            groups = [owner[int(s)] for s in slots] if len(slots) else [direct[q]]
            for us in groups:
                assert sorted(k for _, _, k in us) == list(range(hkv)) and all(o == q for o, _, _ in us)
                ui = us[0][1]
                toff, nt = int(units[ui, 0]), int(units[ui, 1])
                pos = int(d["unit_pos"][ui])
                for k in range(toff, toff + nt):
                    for row in range(int(valid[k])):
                        if pos < vis:
                            seen.append((pos, int(block[k]) * 32 + row))
                        pos += 1
                assert all(np.array_equal(units[ui, :2], units[u2, :2]) and d["unit_pos"][u2] == d["unit_pos"][ui]
                           for _, u2, _ in us)
            seen.sort()
            assert [p for p, _ in seen] == list(range(vis)), (x_sid, j)
            assert [sl for _, sl in seen] == path_slots[:vis]
        r += mq


@pytest.mark.parametrize("flags", [0, tp.TP_MMA_SYNC])
@pytest.mark.parametrize("seed", range(8))
def test_prefill_schedule_covers_each_visible_token_once(seed, flags):
    s = workloads.random_tree(seed=seed, n_prompts=3, max_depth=4, heads=workloads.Heads(8, 2, 64))
    f, ids = metadata_forest(s)
    model = oracle.OracleForest(block_tokens=32).replay(s)
    rng = np.random.default_rng(seed)
    live = [sid for sid in ids if model.nodes[sid].state != "dead" and model.nodes[sid].n_tokens > 0]
    pick = [live[int(i)] for i in rng.integers(0, len(live), min(len(live), 7))]
    counts = [int(rng.integers(0, model.nodes[x].n_tokens + 1)) for x in pick]
    check_prefill_coverage(f, model, ids, pick, counts, flags)


def test_prefill_schedule_long_paths_are_chunked_and_clipped():
    # 1000-token prompt, 600-token segment prefilled whole: several chunks per
    # row block, and early row blocks read fewer tiles than late ones
    s = workloads.single_path(seed=1, lengths=(1000, 600), heads=workloads.Heads(28, 4, 128))
    f, ids = metadata_forest(s)
    model = oracle.OracleForest(block_tokens=32).replay(s)
    leaf = s.leaves[0]
    check_prefill_coverage(f, model, ids, [leaf], [600])
    check_prefill_coverage(f, model, ids, [leaf], [600], tp.TP_MMA_SYNC)
    d = tp.tp_debug_prefill_schedule(f.handle, [ids[leaf]], [600], tp.TP_MMA_SYNC)
    assert d["units"][:, 1].max() <= 128
    first_block = d["units"][d["units"][:, 2] == 0]
    last_block = d["units"][d["units"][:, 2] == d["units"][:, 2].max()]
    assert first_block[:, 1].sum() < last_block[:, 1].sum()


def test_prefill_argument_errors():
    s = workloads.tiny(seed=0)
    f, ids = metadata_forest(s)
    leaf = ids[s.leaves[0]]
    n_tok = f.node_info(leaf)["n_tokens"]
    with pytest.raises(tp.TreepoError):
        tp.tp_debug_prefill_schedule(f.handle, [leaf], [n_tok + 1])
    with pytest.raises(tp.TreepoError):
        tp.tp_debug_prefill_schedule(f.handle, [10 ** 6], [1])
    d = tp.tp_debug_prefill_schedule(f.handle, [leaf], [0])
    assert len(d["units"]) == 0 and len(d["vis"]) == 0
    wide = tp.Forest(128, 1, 64, pool_blocks=16, device=None)       # g = 128 > 64
    r = wide.add_root()
    tp.tp_append_segment(wide.handle, r, 4, None, None)
    with pytest.raises(tp.TreepoError):
        tp.tp_debug_prefill_schedule(wide.handle, [r], [1])
