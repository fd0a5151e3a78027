// forest.cpp -- host side of libtreepo: the paged block pool, node table and
// the tree-walk scheduler that turns a leaf set into attention work units.
//
// Scheduling (the reason the library exists). A decode call names n leaf
// occurrences. Every node on the union of their root-to-leaf paths is read
// once per kv head, with the queries of ALL occurrences below it stacked as
// rows of one tile: the sub-group G_j of trajectories that share the
// predecessor at depth j (Sec. 2.3, Eq. groups) is exactly the row set of the
// node at depth j. A node whose occurrence set equals its parent's is folded
// into the parent's item (a chain of single-branch segments is one item).
// Items are cut into chunks of at most C blocks; each (chunk, kv head) is a
// unit that writes one fp32 partial (normalised o, log2 LSE) per row, and a
// merge pass folds each occurrence's partials by log-sum-exp.
#include <algorithm>
#include <cstring>

#include "forest.h"

namespace tp {

// ---------------------------------------------------------------- pool ---
void BlockPool::init(int64_t n_blocks) {
    n_ = n_blocks;
    free_ = n_blocks;
    hint_ = 0;
    bits_.assign((size_t)((n_blocks + 63) / 64), ~0ull);
    if (n_blocks % 64) bits_.back() = (1ull << (n_blocks % 64)) - 1;
}

bool BlockPool::alloc(int64_t count, std::vector<int32_t>& out) {
    if (count > free_) return false;
    int64_t w = hint_;
    int64_t got = 0;
    while (got < count) {
        uint64_t word = bits_[(size_t)w];
        while (word && got < count) {
            int b = __builtin_ctzll(word);
            word &= word - 1;
            bits_[(size_t)w] &= ~(1ull << b);
            out.push_back((int32_t)(w * 64 + b));
            ++got;
        }
        if (got < count) ++w;
    }
    hint_ = w;
    free_ -= count;
    return true;
}

void BlockPool::release(const std::vector<int32_t>& blocks) {
    for (int32_t b : blocks) {
        bits_[(size_t)(b / 64)] |= 1ull << (b % 64);
        hint_ = std::min<int64_t>(hint_, b / 64);
    }
    free_ += (int64_t)blocks.size();
}

// ------------------------------------------------------------- helpers ---
tp_status fail(tp_tree* t, tp_status code, const std::string& msg) {
    if (t) t->err = msg;
    return code;
}

tp_status check_live(tp_tree* t, tp_node node, bool need_leaf) {
    if (node < 0 || node >= (tp_node)t->nodes.size())
        return fail(t, TP_ERR_BAD_NODE, "unknown node id " + std::to_string(node));
    const Node& nd = t->nodes[(size_t)node];
    if (nd.state == 2) return fail(t, TP_ERR_BAD_NODE, "node " + std::to_string(node) + " was pruned");
    if (need_leaf && nd.state != 0)
        return fail(t, TP_ERR_NOT_LEAF, "node " + std::to_string(node) + " is an interior node");
    return TP_OK;
}

static inline int32_t tile_word(int32_t block, int32_t valid) {
    return (block << kTileValidBits) | (valid - 1);
}

static void node_tiles(const tp_tree* t, const Node& nd, std::vector<int32_t>& tiles) {
    const int32_t bt = t->cfg.block_tokens;
    const int32_t nb = (int32_t)nd.blocks.size();
    for (int32_t b = 0; b < nb; ++b) {
        int32_t valid = (b + 1 < nb) ? bt : nd.n_tokens - b * bt;
        tiles.push_back(tile_word(nd.blocks[(size_t)b], valid));
    }
}

void path_tiles(const tp_tree* t, tp_node leaf, std::vector<int32_t>& tiles) {
    std::vector<int32_t> chain;
    for (int32_t x = leaf; x != -1; x = t->nodes[(size_t)x].parent) chain.push_back(x);
    for (size_t k = chain.size(); k-- > 0;) node_tiles(t, t->nodes[(size_t)chain[k]], tiles);
}

// ------------------------------------------------------------ schedule ---
namespace {
struct Item {
    int32_t occ_off;  // into the occ vector
    int32_t n_occ;
    int32_t tile_off;  // into the tiles vector
    int32_t n_tiles;
};
constexpr int64_t kTargetUnits = 152 * 2 * 6;  // SMs x resident CTAs x waves
constexpr int32_t kMinChunkTiles = 4;
constexpr int32_t kMaxChunkTiles = 64;
}  // namespace

tp_status build_schedule(tp_tree* t, const tp_node* leaves, int32_t n, uint32_t flags, Schedule& S) {
    const int32_t hq = t->cfg.num_q_heads, hkv = t->cfg.num_kv_heads, g = hq / hkv;
    const bool share = !(flags & TP_DECODE_NO_SHARE);
    const bool cuda_core_small = (flags & TP_DECODE_CUDA_CORE_SMALL) != 0;
    const bool all_tc = (flags & TP_DECODE_ALL_TCGEN05) != 0;
    const bool use_tc = all_tc || (flags & TP_DECODE_TCGEN05) != 0;
    for (int32_t i = 0; i < n; ++i) {
        tp_status st = check_live(t, leaves[i], true);
        if (st != TP_OK) return st;
        const Node& nd = t->nodes[(size_t)leaves[i]];
        if (nd.path_before + nd.n_tokens == 0)
            return fail(t, TP_ERR_EMPTY_PATH, "leaf " + std::to_string(leaves[i]) + " has no token on its path");
    }

    std::vector<Item> items;
    std::vector<int32_t> occ, tiles;
    if (share) {
        // 1. nodes on the union of the paths, with their occurrence counts
        const size_t nn = t->nodes.size();
        if (t->mark.size() < nn) {
            t->mark.resize(nn, 0);
            t->local.resize(nn, 0);
        }
        if (++t->epoch == 0) {
            std::fill(t->mark.begin(), t->mark.end(), 0u);
            t->epoch = 1;
        }
        std::vector<int32_t> touched, cnt;
        for (int32_t i = 0; i < n; ++i) {
            for (int32_t x = leaves[i]; x != -1; x = t->nodes[(size_t)x].parent) {
                if (t->mark[(size_t)x] != t->epoch) {
                    t->mark[(size_t)x] = t->epoch;
                    t->local[(size_t)x] = (int32_t)touched.size();
                    touched.push_back(x);
                    cnt.push_back(0);
                }
                ++cnt[(size_t)t->local[(size_t)x]];
            }
        }
        // 2. occurrence list of every touched node (ascending occurrence)
        std::vector<int32_t> start(touched.size() + 1, 0), fill(touched.size(), 0), all_occ;
        for (size_t k = 0; k < touched.size(); ++k) start[k + 1] = start[k] + cnt[k];
        all_occ.resize((size_t)start.back());
        for (int32_t i = 0; i < n; ++i)
            for (int32_t x = leaves[i]; x != -1; x = t->nodes[(size_t)x].parent) {
                int32_t k = t->local[(size_t)x];
                all_occ[(size_t)(start[(size_t)k] + fill[(size_t)k]++)] = i;
            }
        // 3. chains: ids ascend from parent to child, so ascending id order
        //    visits every parent before its children
        std::vector<int32_t> order(touched);
        std::sort(order.begin(), order.end());
        std::vector<int32_t> item_of(touched.size(), -1);
        std::vector<std::vector<int32_t>> item_nodes;
        for (int32_t x : order) {
            const int32_t k = t->local[(size_t)x];
            const int32_t p = t->nodes[(size_t)x].parent;
            int32_t it;
            if (p != -1 && cnt[(size_t)t->local[(size_t)p]] == cnt[(size_t)k]) {
                it = item_of[(size_t)t->local[(size_t)p]];  // same occurrence set: extend
            } else {
                it = (int32_t)items.size();
                items.push_back({(int32_t)occ.size(), cnt[(size_t)k], 0, 0});
                occ.insert(occ.end(), all_occ.begin() + start[(size_t)k], all_occ.begin() + start[(size_t)k + 1]);
                item_nodes.emplace_back();
            }
            item_of[(size_t)k] = it;
            item_nodes[(size_t)it].push_back(x);
        }
        for (size_t it = 0; it < items.size(); ++it) {
            items[it].tile_off = (int32_t)tiles.size();
            for (int32_t x : item_nodes[it]) node_tiles(t, t->nodes[(size_t)x], tiles);
            items[it].n_tiles = (int32_t)tiles.size() - items[it].tile_off;
        }
    } else {
        // every occurrence reads its whole path on its own
        for (int32_t i = 0; i < n; ++i) {
            Item it{(int32_t)occ.size(), 1, (int32_t)tiles.size(), 0};
            occ.push_back(i);
            path_tiles(t, leaves[i], tiles);
            it.n_tiles = (int32_t)tiles.size() - it.tile_off;
            items.push_back(it);
        }
    }

    // 4. chunk size: enough units to fill the GPU several times over, but
    //    every chunk of an item costs one fp32 partial per stacked row
    //    ((head_dim + 1) * 4 bytes written, then read by the merge); an item
    //    with R rows per kv head is cut no finer than 1.25 R blocks, which
    //    keeps that traffic under ~5% of the chunk's KV bytes.
    int64_t work = 0;
    for (const Item& it : items) work += (int64_t)it.n_tiles * hkv;
    const int32_t chunk = (int32_t)std::min<int64_t>(
        kMaxChunkTiles, std::max<int64_t>(kMinChunkTiles, (work + kTargetUnits - 1) / kTargetUnits));

    // 5. units, partial slots and merge entries
    std::vector<int32_t> tc_units, tensor_units, small_units;
    std::vector<int32_t> pair_occ, pair_slot;  // merge entries before sorting
    int32_t n_slots = 0;
    for (const Item& it : items) {
        if (it.n_tiles == 0) continue;
        const int32_t rows_chunk = (it.n_occ * g * 5 + 3) / 4;
        const int32_t n_chunks =
            std::max(rows_chunk > chunk ? std::max(1, it.n_tiles / rows_chunk) : (it.n_tiles + chunk - 1) / chunk,
                     (it.n_tiles + kMaxUnitTiles - 1) / kMaxUnitTiles);
        const int32_t base = it.n_tiles / n_chunks, extra = it.n_tiles % n_chunks;
        const int32_t rows = it.n_occ * g;
        int32_t toff = it.tile_off;
        for (int32_t c = 0; c < n_chunks; ++c) {
            const int32_t nt = base + (c < extra ? 1 : 0);
            const int32_t slot_base = n_slots;
            n_slots += it.n_occ;
            for (int32_t p = 0; p < it.n_occ; ++p) {
                pair_occ.push_back(occ[(size_t)(it.occ_off + p)]);
                pair_slot.push_back(slot_base + p);
            }
            for (int32_t h = 0; h < hkv; ++h) {
                if (rows < kTensorMinRows && cuda_core_small) {
                    const int32_t u[kUnitWords] = {toff, nt, it.occ_off, 0, rows, slot_base, h, KIND_CUDA_CORE};
                    small_units.insert(small_units.end(), u, u + kUnitWords);
                } else if (use_tc && (all_tc ? rows >= kTcAnyRows : rows >= kTcMinRows && nt >= kTcMinTiles)) {
                    for (int32_t r0 = 0; r0 < rows; r0 += kTcRowsPerUnit) {
                        const int32_t nr = std::min(kTcRowsPerUnit, rows - r0);
                        const int32_t u[kUnitWords] = {toff, nt, it.occ_off, r0, nr, slot_base, h, KIND_TC};
                        tc_units.insert(tc_units.end(), u, u + kUnitWords);
                    }
                } else {
                    for (int32_t r0 = 0; r0 < rows; r0 += kTensorRowsPerUnit) {
                        const int32_t nr = std::min(kTensorRowsPerUnit, rows - r0);
                        const int32_t u[kUnitWords] = {toff, nt, it.occ_off, r0, nr, slot_base, h, KIND_TENSOR};
                        tensor_units.insert(tensor_units.end(), u, u + kUnitWords);
                    }
                }
            }
            toff += nt;
        }
    }

    // 6. unit order: tcgen05, then mma.sync, then CUDA-core units; longer
    //    units first within a kind
    auto sort_units = [](std::vector<int32_t>& u) {
        const size_t cnt = u.size() / kUnitWords;
        std::vector<int32_t> idx(cnt);
        for (size_t k = 0; k < cnt; ++k) idx[k] = (int32_t)k;
        std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) {
            return u[(size_t)a * kUnitWords + U_N_TILES] > u[(size_t)b * kUnitWords + U_N_TILES];
        });
        std::vector<int32_t> out(u.size());
        for (size_t k = 0; k < cnt; ++k)
            std::memcpy(&out[k * kUnitWords], &u[(size_t)idx[k] * kUnitWords], sizeof(int32_t) * kUnitWords);
        u.swap(out);
    };
    sort_units(tc_units);
    sort_units(tensor_units);
    sort_units(small_units);

    // 7. merge CSR by occurrence (stable: root-first slot order per leaf)
    std::vector<int32_t> merge_off((size_t)n + 1, 0), merge_slot(pair_occ.size());
    for (int32_t i : pair_occ) ++merge_off[(size_t)i + 1];
    for (int32_t i = 0; i < n; ++i) merge_off[(size_t)i + 1] += merge_off[(size_t)i];
    {
        std::vector<int32_t> pos(merge_off.begin(), merge_off.end() - 1);
        for (size_t k = 0; k < pair_occ.size(); ++k) merge_slot[(size_t)pos[(size_t)pair_occ[k]]++] = pair_slot[k];
    }

    // 8. assemble
    S.n_tc = (int32_t)(tc_units.size() / kUnitWords);
    S.n_tensor = (int32_t)(tensor_units.size() / kUnitWords);
    S.n_units = S.n_tc + S.n_tensor + (int32_t)(small_units.size() / kUnitWords);
    S.n_tiles = (int32_t)tiles.size();
    S.n_occ = (int32_t)occ.size();
    S.n = n;
    S.n_slots = n_slots;
    S.n_merge = (int32_t)merge_slot.size();
    S.off_units = kSchedHeaderWords;
    S.off_tiles = S.off_units + (int64_t)S.n_units * kUnitWords;
    S.off_occ = S.off_tiles + S.n_tiles;
    S.off_merge_off = S.off_occ + S.n_occ;
    S.off_merge_slot = S.off_merge_off + n + 1;
    const int64_t total = S.off_merge_slot + S.n_merge;
    if (total >= (int64_t)1 << 31) return fail(t, TP_ERR_INVALID_ARG, "schedule too large");
    S.words.assign((size_t)total, 0);
    int32_t* w = S.words.data();
    w[0] = kSchedMagic;
    w[1] = S.n_units;
    w[2] = S.n_tiles;
    w[3] = S.n_occ;
    w[4] = n;
    w[5] = S.n_slots;
    w[6] = S.n_merge;
    w[7] = g;
    w[8] = S.n_tensor;
    w[9] = S.n_tc;
    std::copy(tc_units.begin(), tc_units.end(), w + S.off_units);
    std::copy(tensor_units.begin(), tensor_units.end(), w + S.off_units + tc_units.size());
    std::copy(small_units.begin(), small_units.end(), w + S.off_units + tc_units.size() + tensor_units.size());
    std::copy(tiles.begin(), tiles.end(), w + S.off_tiles);
    std::copy(occ.begin(), occ.end(), w + S.off_occ);
    std::copy(merge_off.begin(), merge_off.end(), w + S.off_merge_off);
    std::copy(merge_slot.begin(), merge_slot.end(), w + S.off_merge_slot);
    return TP_OK;
}

}  // namespace tp
