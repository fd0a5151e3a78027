"""The bounds-checked build's index predicates, on the host (no GPU).

libtreepo_checked.so compiles the kernels with TP_BOUNDS_CHECK: before each
access they check the schedule words they index with and, on a failed
check, skip the access and flag the error (tp_sync reports it). The same
predicates run on the host through tp_debug_check_schedule. Here every
schedule the library builds passes them, and a schedule with one planted
bad word -- each kind of index the kernels take -- is caught in the right
category. The planted words never reach a GPU.
"""
import os
import re
import subprocess

import numpy as np
import pytest

import paper_2508_17445_gb300 as tp
import workloads

HDR = 16          # schedule header words
UW = 8            # unit words
U_TILE_OFF, U_N_TILES, U_OCC_OFF, U_ROW0, U_N_ROWS, U_SLOT_BASE, U_KVH, U_KIND = range(8)


def meta_tree(script, pool_extra=8):
    h = script.heads
    f = tp.Forest(h.num_q_heads, h.num_kv_heads, h.head_dim, pool_blocks=script.upper_bound_blocks(32) + pool_extra,
                  device=None)
    ids = f.replay(script.ops)
    return f, ids


def sections(w):
    n_units, n_tiles, n_occ, n, n_slots, n_merge = (int(x) for x in w[1:7])
    off_tiles = HDR + UW * n_units
    off_occ = off_tiles + n_tiles
    off_moff = off_occ + n_occ
    off_mslot = off_moff + n + 1
    return dict(n_units=n_units, n_tiles=n_tiles, n_occ=n_occ, n=n, n_slots=n_slots, n_merge=n_merge,
                off_tiles=off_tiles, off_occ=off_occ, off_moff=off_moff, off_mslot=off_mslot)


FLAG_SETS = [0, tp.TP_DECODE_CUDA_CORE_SMALL, tp.TP_DECODE_NO_SHARE, tp.TP_MMA_SYNC, tp.TP_DECODE_TCGEN05]


@pytest.mark.parametrize("seed", range(3))
def test_library_schedules_pass_every_check(seed):
    s = workloads.random_tree(seed=seed, heads=workloads.Heads(28, 4, 128), n_prompts=3, max_depth=5,
                              prompt_range=(1, 400), seg_range=(1, 200))
    f, ids = meta_tree(s)
    leaves = [ids[x] for x in s.leaves]
    zero = dict.fromkeys(tp.CHECK_CATEGORIES, 0)
    for flags in FLAG_SETS:
        w = tp.tp_debug_schedule(f.handle, leaves, flags)["words"]
        assert tp.tp_debug_check_schedule(f.handle, w) == zero, flags
    # prefill schedules (direct-write units with slot_base -1 are legal there)
    nodes = [ids[x] for x in s.leaves[:4]]
    counts = [min(40, f.node_info(x)["n_tokens"]) for x in nodes]
    for flags in (0, tp.TP_MMA_SYNC):
        w = tp.tp_debug_prefill_schedule(f.handle, nodes, counts, flags)["words"]
        assert tp.tp_debug_check_schedule(f.handle, w) == zero, flags
    f.close()


def _decode_words(flags=0):
    s = workloads.qwen7b(seed=2, n_prompts=2)
    f, ids = meta_tree(s)
    w = tp.tp_debug_schedule(f.handle, [ids[x] for x in s.leaves], flags)["words"].copy()
    return f, w


def _unit_of_kind(w, kind):
    n_units = int(w[1])
    for k in range(n_units):
        if w[HDR + UW * k + U_KIND] == kind:
            return HDR + UW * k
    raise AssertionError(f"no unit of kind {kind}")


def plant(name, w, pool_blocks, hkv):
    """One bad word of the given kind; returns the category it must be caught in."""
    x = sections(w)
    u_tc = _unit_of_kind(w, 2)
    u_mma = _unit_of_kind(w, 1)
    if name == "tile_block_past_pool":
        w[x["off_tiles"] + 3] = (pool_blocks << 7) | 31
        return "tiles"
    if name == "tile_too_many_tokens":
        w[x["off_tiles"] + 5] = (int(w[x["off_tiles"] + 5]) & ~127) | 40
        return "tiles"
    if name == "tile_negative":
        w[x["off_tiles"]] = -5
        return "tiles"
    if name == "unit_tiles_past_section":
        w[u_tc + U_TILE_OFF] = x["n_tiles"] - 1
        w[u_tc + U_N_TILES] = 2
        return "units"
    if name == "unit_too_long":
        w[u_mma + U_N_TILES] = 129
        return "units"
    if name == "unit_kv_head":
        w[u_mma + U_KVH] = hkv
        return "units"
    if name == "unit_rows_past_kind":
        w[u_mma + U_N_ROWS] = 65                  # an mma.sync unit holds 64 rows at most
        return "units"
    if name == "unit_occurrences_past_list":
        w[u_tc + U_OCC_OFF] = x["n_occ"] - 1
        return "units"
    if name == "unit_slot_past_partials":
        w[u_tc + U_SLOT_BASE] = x["n_slots"] - 1
        return "units"
    if name == "unit_direct_write_in_decode":
        w[u_tc + U_SLOT_BASE] = -1                # only prefill units write O directly
        return "units"
    if name == "unit_kind_out_of_order":
        w[u_tc + U_KIND] = 1
        return "units"
    if name == "occurrence_past_rows":
        w[x["off_occ"] + 2] = x["n"]
        return "occ"
    if name == "merge_range_backwards":
        i = 3
        w[x["off_moff"] + i], w[x["off_moff"] + i + 1] = w[x["off_moff"] + i + 1] + 1, w[x["off_moff"] + i]
        return "merge_ranges"
    if name == "merge_range_past_list":
        w[x["off_moff"] + x["n"]] = x["n_merge"] + 1
        return "merge_ranges"
    if name == "merge_slot_past_partials":
        w[x["off_mslot"] + 7] = x["n_slots"]
        return "merge_slots"
    off_mrec = x["off_mslot"] + x["n_merge"]
    if name == "merge_record_count_wrong":
        w[off_mrec + 16 * 3] += 1
        return "merge_ranges"
    if name == "merge_record_slot_past_partials":
        w[off_mrec + 16 * 5 + 1] = x["n_slots"]
        return "merge_slots"
    raise ValueError(name)


PLANTS = ["tile_block_past_pool", "tile_too_many_tokens", "tile_negative", "unit_tiles_past_section",
          "unit_too_long", "unit_kv_head", "unit_rows_past_kind", "unit_occurrences_past_list",
          "unit_slot_past_partials", "unit_direct_write_in_decode", "unit_kind_out_of_order",
          "occurrence_past_rows", "merge_range_backwards", "merge_range_past_list", "merge_slot_past_partials",
          "merge_record_count_wrong", "merge_record_slot_past_partials"]


@pytest.mark.parametrize("name", PLANTS)
def test_each_planted_bad_word_is_caught(name):
    f, w = _decode_words()
    assert sum(tp.tp_debug_check_schedule(f.handle, w).values()) == 0
    want = plant(name, w, f.cfg.pool_blocks, f.cfg.num_kv_heads)
    got = tp.tp_debug_check_schedule(f.handle, w)
    assert got[want] >= 1, (name, got)
    assert all(v == 0 for k, v in got.items() if k not in (want, "merge_ranges")), (name, got)
    f.close()


def test_not_a_schedule_is_rejected():
    f, w = _decode_words()
    bad = w.copy()
    bad[0] = 0
    with pytest.raises(tp.TreepoError) as e:
        tp.tp_debug_check_schedule(f.handle, bad)
    assert e.value.code == "INVALID_ARG"
    with pytest.raises(tp.TreepoError):
        tp.tp_debug_check_schedule(f.handle, w[: len(w) // 2])   # shorter than its header says
    f.close()


def test_checked_library_builds_with_the_same_calls():
    from paper_2508_17445_gb300 import build
    path = build.build(checked=True)
    assert os.path.basename(path) == "libtreepo_checked.so"
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (tp_\w+)", out))
    assert set(tp.EXPORTED_SYMBOLS) <= exported
