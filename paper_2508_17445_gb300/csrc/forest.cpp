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
    if (nb == 0) return;
    const size_t off = tiles.size();
    tiles.resize(off + (size_t)nb);
    int32_t* dst = tiles.data() + off;
    const int32_t* src = nd.blocks.data();
    for (int32_t b = 0; b < nb; ++b) dst[b] = tile_word(src[b], bt);
    dst[nb - 1] = tile_word(src[nb - 1], nd.n_tokens - (nb - 1) * bt);
}

void path_tiles(const tp_tree* t, tp_node leaf, std::vector<int32_t>& tiles) {
    std::vector<int32_t> chain;
    for (int32_t x = leaf; x != -1; x = t->nodes[(size_t)x].parent) chain.push_back(x);
    for (size_t k = chain.size(); k-- > 0;) node_tiles(t, t->nodes[(size_t)chain[k]], tiles);
}

// ------------------------------------------------------------ schedule ---
namespace {
constexpr int64_t kTargetUnits = 152 * 2 * 6;  // SMs x resident CTAs x waves
constexpr int32_t kMinChunkTiles = 4;
constexpr int32_t kMaxChunkTiles = 64;

// Stable reorder of unit records (`width` words, n_tiles in word
// U_N_TILES) longest first (a counting sort: n_tiles <= kMaxUnitTiles).
void sort_units(std::vector<int32_t>& u, std::vector<int32_t>& out, std::vector<int32_t>& bucket,
                size_t width = kUnitWords) {
    const size_t cnt = u.size() / width;
    if (cnt < 2) return;
    bucket.assign(kMaxUnitTiles + 2, 0);
    for (size_t k = 0; k < cnt; ++k) ++bucket[(size_t)(kMaxUnitTiles - u[k * width + U_N_TILES] + 1)];
    for (int b = 1; b < kMaxUnitTiles + 2; ++b) bucket[(size_t)b] += bucket[(size_t)b - 1];
    out.resize(u.size());
    for (size_t k = 0; k < cnt; ++k) {
        const int32_t pos = bucket[(size_t)(kMaxUnitTiles - u[k * width + U_N_TILES])]++;
        std::memcpy(&out[(size_t)pos * width], &u[k * width], sizeof(int32_t) * width);
    }
    u.swap(out);
}

// Merge CSR by occurrence from (occurrence, slot) pairs, stable.
void merge_csr(SchedScratch& X, int32_t n) {
    X.merge_off.assign((size_t)n + 1, 0);
    X.merge_slot.resize(X.pair_occ.size());
    for (int32_t i : X.pair_occ) ++X.merge_off[(size_t)i + 1];
    for (int32_t i = 0; i < n; ++i) X.merge_off[(size_t)i + 1] += X.merge_off[(size_t)i];
    X.merge_pos.assign(X.merge_off.begin(), X.merge_off.end() - 1);
    for (size_t k = 0; k < X.pair_occ.size(); ++k)
        X.merge_slot[(size_t)X.merge_pos[(size_t)X.pair_occ[k]]++] = X.pair_slot[k];
}

// Fixed-size merge records from the CSR: [count, slots..., 0...], or
// [-1, 0...] for an occurrence with more than kMergeRecWords - 1 slots.
void merge_records(const SchedScratch& X, int32_t n, int32_t* rec) {
    std::fill(rec, rec + (int64_t)n * kMergeRecWords, 0);
    for (int32_t i = 0; i < n; ++i) {
        const int32_t beg = X.merge_off[(size_t)i], cnt = X.merge_off[(size_t)i + 1] - beg;
        int32_t* r = rec + (int64_t)i * kMergeRecWords;
        if (cnt >= kMergeRecWords) {
            r[0] = -1;
            continue;
        }
        r[0] = cnt;
        std::copy(X.merge_slot.begin() + beg, X.merge_slot.begin() + beg + cnt, r + 1);
    }
}
}  // namespace

tp_status build_schedule(tp_tree* t, const tp_node* leaves, int32_t n, uint32_t flags, Schedule& S) {
    const int32_t hq = t->cfg.num_q_heads, hkv = t->cfg.num_kv_heads, g = hq / hkv;
    const bool share = !(flags & TP_DECODE_NO_SHARE);
    const bool cuda_core_small = (flags & TP_DECODE_CUDA_CORE_SMALL) != 0;
    for (int32_t i = 0; i < n; ++i) {
        tp_status st = check_live(t, leaves[i], true);
        if (st != TP_OK) return st;
        const Node& nd = t->nodes[(size_t)leaves[i]];
        if (nd.path_before + nd.n_tokens == 0)
            return fail(t, TP_ERR_EMPTY_PATH, "leaf " + std::to_string(leaves[i]) + " has no token on its path");
    }

    SchedScratch& X = t->scratch;
    std::vector<Item>& items = X.items;
    std::vector<int32_t>& occ = X.occ;
    std::vector<int32_t>& tiles = X.tiles;
    items.clear();
    occ.clear();
    tiles.clear();
    X.tail_node.clear();
    X.tail_tile.clear();
    // a leaf's last tile: recorded when its last block is partly filled,
    // since only then can an append leave the block list unchanged
    auto note_tail = [&](const Node& nd, int32_t leaf) {
        if (!nd.blocks.empty() && nd.n_tokens % t->cfg.block_tokens) {
            X.tail_node.push_back(leaf);
            X.tail_tile.push_back((int32_t)tiles.size() - 1);
        }
    };
    if (share) {
        // 1. nodes on the union of the paths, with their occurrence counts
        const size_t nn = t->nodes.size();
        if (X.mark.size() < nn) {
            X.mark.resize(nn, 0);
            X.local.resize(nn, 0);
        }
        if (++X.epoch == 0) {
            std::fill(X.mark.begin(), X.mark.end(), 0u);
            X.epoch = 1;
        }
        std::vector<int32_t>& touched = X.touched;
        std::vector<int32_t>& cnt = X.cnt;
        touched.clear();
        cnt.clear();
        for (int32_t i = 0; i < n; ++i) {
            for (int32_t x = leaves[i]; x != -1; x = t->nodes[(size_t)x].parent) {
                if (X.mark[(size_t)x] != X.epoch) {
                    X.mark[(size_t)x] = X.epoch;
                    X.local[(size_t)x] = (int32_t)touched.size();
                    touched.push_back(x);
                    cnt.push_back(0);
                }
                ++cnt[(size_t)X.local[(size_t)x]];
            }
        }
        // 2. occurrence list of every touched node (ascending occurrence)
        const size_t nt = touched.size();
        X.start.assign(nt + 1, 0);
        X.fill.assign(nt, 0);
        for (size_t k = 0; k < nt; ++k) X.start[k + 1] = X.start[k] + cnt[k];
        X.all_occ.resize((size_t)X.start.back());
        for (int32_t i = 0; i < n; ++i)
            for (int32_t x = leaves[i]; x != -1; x = t->nodes[(size_t)x].parent) {
                const int32_t k = X.local[(size_t)x];
                X.all_occ[(size_t)(X.start[(size_t)k] + X.fill[(size_t)k]++)] = i;
            }
        // 3. chains: ids ascend from parent to child, so ascending id order
        //    visits every parent before its children
        X.order.assign(touched.begin(), touched.end());
        std::sort(X.order.begin(), X.order.end());
        X.item_of.assign(nt, -1);
        X.item_cnt.clear();
        for (int32_t x : X.order) {
            const int32_t k = X.local[(size_t)x];
            const int32_t p = t->nodes[(size_t)x].parent;
            int32_t it;
            if (p != -1 && cnt[(size_t)X.local[(size_t)p]] == cnt[(size_t)k]) {
                it = X.item_of[(size_t)X.local[(size_t)p]];  // same occurrence set: extend
            } else {
                it = (int32_t)items.size();
                items.push_back({(int32_t)occ.size(), cnt[(size_t)k], 0, 0});
                occ.insert(occ.end(), X.all_occ.begin() + X.start[(size_t)k], X.all_occ.begin() + X.start[(size_t)k + 1]);
                X.item_cnt.push_back(0);
            }
            X.item_of[(size_t)k] = it;
            ++X.item_cnt[(size_t)it];
        }
        // nodes of each item in ascending id order (CSR)
        const size_t ni = items.size();
        X.item_start.assign(ni + 1, 0);
        for (size_t it = 0; it < ni; ++it) X.item_start[it + 1] = X.item_start[it] + X.item_cnt[it];
        X.item_nodes.resize(nt);
        X.fill.assign(ni, 0);
        for (int32_t x : X.order) {
            const int32_t it = X.item_of[(size_t)X.local[(size_t)x]];
            X.item_nodes[(size_t)(X.item_start[(size_t)it] + X.fill[(size_t)it]++)] = x;
        }
        for (size_t it = 0; it < ni; ++it) {
            items[it].tile_off = (int32_t)tiles.size();
            for (int32_t k = X.item_start[it]; k < X.item_start[it + 1]; ++k) {
                const int32_t x = X.item_nodes[(size_t)k];
                const Node& nd = t->nodes[(size_t)x];
                node_tiles(t, nd, tiles);
                if (nd.state == 0) note_tail(nd, x);
            }
            items[it].n_tiles = (int32_t)tiles.size() - items[it].tile_off;
        }
    } else {
        // every occurrence reads its whole path on its own
        for (int32_t i = 0; i < n; ++i) {
            Item it{(int32_t)occ.size(), 1, (int32_t)tiles.size(), 0};
            occ.push_back(i);
            path_tiles(t, leaves[i], tiles);
            note_tail(t->nodes[(size_t)leaves[i]], leaves[i]);
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
    // tcgen05 for every unit of more than one 16-row MMA tile unless
    // TP_MMA_SYNC; TP_DECODE_TCGEN05 alone keeps it to long, tall chunks. A
    // call reading less than kSmallCallBytes of K/V is bound by launch
    // latency: its stacked rows stay on mma.sync, so the whole call is one
    // attention kernel on the tree's stream, without the tcgen05 kernel's
    // side-stream fork and join (TP_DECODE_ALL_TCGEN05 still forces tcgen05).
    const int64_t tile_bytes = (int64_t)t->cfg.block_tokens * t->cfg.head_dim * 2 * 2;
    const bool small_call = work * tile_bytes < kSmallCallBytes && !(flags & TP_DECODE_ALL_TCGEN05);
    const bool use_tc = (flags & TP_MMA_SYNC) == 0 && !small_call;
    const bool all_tc = use_tc && !((flags & TP_DECODE_TCGEN05) && !(flags & TP_DECODE_ALL_TCGEN05));

    // 5. units, partial slots and merge entries
    std::vector<int32_t>& tc_units = X.units[0];
    std::vector<int32_t>& tensor_units = X.units[1];
    std::vector<int32_t>& small_units = X.units[2];
    std::vector<int32_t>& pair_occ = X.pair_occ;
    std::vector<int32_t>& pair_slot = X.pair_slot;
    tc_units.clear();
    tensor_units.clear();
    small_units.clear();
    pair_occ.clear();
    pair_slot.clear();
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
            // one unit per (kv head, block of rows); the kind depends only on
            // the chunk's rows and length
            int32_t kind, rpu;
            if (rows < kTensorMinRows && cuda_core_small) {
                kind = KIND_CUDA_CORE;
                rpu = rows;
            } else if (use_tc && (all_tc ? rows >= kTcAnyRows : rows >= kTcMinRows && nt >= kTcMinTiles)) {
                kind = KIND_TC;
                rpu = kTcRowsPerUnit;
            } else {
                kind = KIND_TENSOR;
                rpu = kTensorRowsPerUnit;
            }
            std::vector<int32_t>& dst = kind == KIND_TC ? tc_units : kind == KIND_TENSOR ? tensor_units : small_units;
            const int32_t row_blocks = (rows + rpu - 1) / rpu;
            const size_t at = dst.size();
            dst.resize(at + (size_t)hkv * row_blocks * kUnitWords);
            int32_t* u = dst.data() + at;
            for (int32_t h = 0; h < hkv; ++h)
                for (int32_t r0 = 0; r0 < rows; r0 += rpu, u += kUnitWords) {
                    u[U_TILE_OFF] = toff;
                    u[U_N_TILES] = nt;
                    u[U_OCC_OFF] = it.occ_off;
                    u[U_ROW0] = r0;
                    u[U_N_ROWS] = std::min(rpu, rows - r0);
                    u[U_SLOT_BASE] = slot_base;
                    u[U_KVH] = h;
                    u[U_KIND] = kind;
                }
            toff += nt;
        }
    }

    // 6. unit order: tcgen05, then mma.sync, then CUDA-core units; longer
    //    units first within a kind
    for (auto& u : X.units) sort_units(u, X.sorted, X.bucket);

    // 7. merge CSR by occurrence (stable: root-first slot order per leaf)
    merge_csr(X, n);
    std::vector<int32_t>& merge_off = X.merge_off;
    std::vector<int32_t>& merge_slot = X.merge_slot;

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
    S.off_merge_rec = S.off_merge_slot + S.n_merge;
    const int64_t total = S.off_merge_rec + (int64_t)n * kMergeRecWords;
    if (total >= (int64_t)1 << 31) return fail(t, TP_ERR_INVALID_ARG, "schedule too large");
    S.words.resize((size_t)total);
    int32_t* w = S.words.data();
    std::fill(w, w + kSchedHeaderWords, 0);
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
    w[11] = kMergeRecWords;
    std::copy(tc_units.begin(), tc_units.end(), w + S.off_units);
    std::copy(tensor_units.begin(), tensor_units.end(), w + S.off_units + tc_units.size());
    std::copy(small_units.begin(), small_units.end(), w + S.off_units + tc_units.size() + tensor_units.size());
    std::copy(tiles.begin(), tiles.end(), w + S.off_tiles);
    std::copy(occ.begin(), occ.end(), w + S.off_occ);
    std::copy(merge_off.begin(), merge_off.end(), w + S.off_merge_off);
    std::copy(merge_slot.begin(), merge_slot.end(), w + S.off_merge_slot);
    merge_records(X, n, w + S.off_merge_rec);
    S.leaf_tail.resize(2 * X.tail_node.size());
    for (size_t k = 0; k < X.tail_node.size(); ++k) {
        S.leaf_tail[2 * k] = X.tail_node[k];
        S.leaf_tail[2 * k + 1] = (int32_t)S.off_tiles + X.tail_tile[k];
    }
    S.prefill = false;
    // With the default routing the mma.sync / CUDA-core kernel (the only one
    // that uses this) gets single-leaf groups of at most 16 rows, one unit per
    // (block, kv head); the no-share control and the other routings give it
    // units that read the same blocks.
    S.kv_read_once = !(flags & (TP_DECODE_NO_SHARE | TP_DECODE_TCGEN05 | TP_MMA_SYNC));
    S.off_unit_pos = S.off_vis = 0;
    return TP_OK;
}

tp_status build_prefill_schedule(tp_tree* t, const tp_node* nodes, const int32_t* m, int32_t n, uint32_t flags,
                                 Schedule& S) {
    const int32_t hq = t->cfg.num_q_heads, hkv = t->cfg.num_kv_heads, g = hq / hkv;
    if (g > kTensorRowsPerUnit)
        return fail(t, TP_ERR_INVALID_ARG, "prefill needs num_q_heads / num_kv_heads <= 64");
    int64_t n_q = 0;
    for (int32_t i = 0; i < n; ++i) {
        tp_status st = check_live(t, nodes[i], false);
        if (st != TP_OK) return st;
        const Node& nd = t->nodes[(size_t)nodes[i]];
        if (m[i] < 0 || m[i] > nd.n_tokens)
            return fail(t, TP_ERR_INVALID_ARG,
                        "n_queries of node " + std::to_string(nodes[i]) + " must lie in [0, its token count]");
        n_q += m[i];
    }
    if (n_q >= (int64_t)1 << 28) return fail(t, TP_ERR_INVALID_ARG, "too many query tokens in one call");
    SchedScratch& X = t->scratch;
    const bool use_tc = !(flags & TP_MMA_SYNC);  // tcgen05 unless asked otherwise (measured faster)
    const int32_t occ_per_block = (use_tc ? kTcRowsPerUnit : kTensorRowsPerUnit) / g;  // whole GQA groups
    // path tiles of every listed node, with each tile's path position
    X.tiles.clear();
    X.tile_pos.clear();
    X.node_tile_off.assign((size_t)n + 1, 0);
    X.vis.resize((size_t)n_q);
    int64_t work = 0;
    for (int32_t i = 0, q0 = 0; i < n; q0 += m[i], ++i) {
        X.node_tile_off[(size_t)i] = (int32_t)X.tiles.size();
        const size_t first = X.tiles.size();
        path_tiles(t, nodes[i], X.tiles);
        int32_t pos = 0;
        for (size_t k = first; k < X.tiles.size(); ++k) {
            X.tile_pos.push_back(pos);
            pos += (X.tiles[k] & ((1 << kTileValidBits) - 1)) + 1;
        }
        const Node& nd = t->nodes[(size_t)nodes[i]];
        const int32_t first_vis = (int32_t)(nd.path_before + nd.n_tokens - m[i]) + 1;
        for (int32_t o = 0; o < m[i]; ++o) X.vis[(size_t)(q0 + o)] = first_vis + o;
        for (int32_t o0 = 0; o0 < m[i]; o0 += occ_per_block) {
            const int32_t o1 = std::min(m[i], o0 + occ_per_block);
            const int32_t lim = X.vis[(size_t)(q0 + o1 - 1)];
            const int32_t* tp0 = X.tile_pos.data() + first;
            work += (int64_t)(std::lower_bound(tp0, tp0 + (X.tiles.size() - first), lim) - tp0) * hkv;
        }
    }
    X.node_tile_off[(size_t)n] = (int32_t)X.tiles.size();
    const int32_t chunk = (int32_t)std::min<int64_t>(
        kMaxUnitTiles, std::max<int64_t>(kMinChunkTiles, (work + kTargetUnits - 1) / kTargetUnits));

    // units of 9 words while sorting: the 8 unit words and the path position
    constexpr int W = kUnitWords + 1;
    std::vector<int32_t>& recs = X.units[1];
    recs.clear();
    X.pair_occ.clear();
    X.pair_slot.clear();
    int32_t n_slots = 0;
    for (int32_t i = 0, q0 = 0; i < n; q0 += m[i], ++i) {
        const int32_t toff = X.node_tile_off[(size_t)i];
        const int32_t n_path = X.node_tile_off[(size_t)i + 1] - toff;
        const int32_t* tpos = X.tile_pos.data() + toff;
        for (int32_t o0 = 0; o0 < m[i]; o0 += occ_per_block) {
            const int32_t o1 = std::min(m[i], o0 + occ_per_block);
            const int32_t lim = X.vis[(size_t)(q0 + o1 - 1)];
            const int32_t nt = (int32_t)(std::lower_bound(tpos, tpos + n_path, lim) - tpos);  // causal clip
            const int32_t n_chunks = (nt + chunk - 1) / chunk;
            const int32_t base = nt / n_chunks, extra = nt % n_chunks;
            for (int32_t c = 0, t0 = 0; c < n_chunks; ++c) {
                const int32_t len = base + (c < extra ? 1 : 0);
                int32_t slot_base = -1;  // one chunk: its units write the final O and LSE
                if (n_chunks > 1) {
                    slot_base = n_slots;
                    n_slots += o1 - o0;
                    for (int32_t o = o0; o < o1; ++o)
                        if (X.vis[(size_t)(q0 + o)] > tpos[t0]) {  // the chunk holds tokens this query sees
                            X.pair_occ.push_back(q0 + o);
                            X.pair_slot.push_back(slot_base + o - o0);
                        }
                }
                for (int32_t h = 0; h < hkv; ++h) {
                    const int32_t u[W] = {toff + t0, len, q0 + o0, 0, (o1 - o0) * g, slot_base, h,
                                          use_tc ? KIND_TC : KIND_TENSOR, tpos[t0]};
                    recs.insert(recs.end(), u, u + W);
                }
                t0 += len;
            }
        }
    }
    sort_units(recs, X.sorted, X.bucket, W);
    merge_csr(X, (int32_t)n_q);

    S.prefill = true;
    S.kv_read_once = false;  // the query blocks of a path re-read its K/V
    S.n_units = (int32_t)(recs.size() / W);
    S.n_tc = use_tc ? S.n_units : 0;
    S.n_tensor = use_tc ? 0 : S.n_units;
    S.n_tiles = (int32_t)X.tiles.size();
    S.n_occ = (int32_t)n_q;
    S.n = (int32_t)n_q;
    S.n_slots = n_slots;
    S.n_merge = (int32_t)X.merge_slot.size();
    S.off_units = kSchedHeaderWords;
    S.off_tiles = S.off_units + (int64_t)S.n_units * kUnitWords;
    S.off_occ = S.off_tiles + S.n_tiles;
    S.off_merge_off = S.off_occ + S.n_occ;
    S.off_merge_slot = S.off_merge_off + S.n + 1;
    S.off_unit_pos = S.off_merge_slot + S.n_merge;
    S.off_vis = S.off_unit_pos + S.n_units;
    S.off_merge_rec = 0;  // no merge records: most query rows are written directly, the rest use the CSR
    const int64_t total = S.off_vis + S.n;
    if (total >= (int64_t)1 << 31) return fail(t, TP_ERR_INVALID_ARG, "schedule too large");
    S.words.resize((size_t)total);
    int32_t* w = S.words.data();
    std::fill(w, w + kSchedHeaderWords, 0);
    w[0] = kSchedMagic;
    w[1] = S.n_units;
    w[2] = S.n_tiles;
    w[3] = S.n_occ;
    w[4] = S.n;
    w[5] = S.n_slots;
    w[6] = S.n_merge;
    w[7] = g;
    w[8] = S.n_tensor;
    w[9] = S.n_tc;
    w[10] = 1;  // prefill schedule
    for (int32_t k = 0; k < S.n_units; ++k) {
        std::memcpy(w + S.off_units + (int64_t)k * kUnitWords, &recs[(size_t)k * W], sizeof(int32_t) * kUnitWords);
        w[S.off_unit_pos + k] = recs[(size_t)k * W + kUnitWords];
    }
    std::copy(X.tiles.begin(), X.tiles.end(), w + S.off_tiles);
    for (int32_t q = 0; q < S.n; ++q) w[S.off_occ + q] = q;
    std::copy(X.merge_off.begin(), X.merge_off.end(), w + S.off_merge_off);
    std::copy(X.merge_slot.begin(), X.merge_slot.end(), w + S.off_merge_slot);
    std::copy(X.vis.begin(), X.vis.end(), w + S.off_vis);
    S.leaf_tail.clear();
    return TP_OK;
}

int32_t patch_schedule(const tp_tree* t, Schedule& S, std::vector<int32_t>& changed) {
    changed.clear();
    const int32_t bt = t->cfg.block_tokens;
    for (size_t k = 0; k < S.leaf_tail.size(); k += 2) {
        const Node& nd = t->nodes[(size_t)S.leaf_tail[k]];
        const int32_t nb = (int32_t)nd.blocks.size();
        const int32_t word = tile_word(nd.blocks[(size_t)nb - 1], nd.n_tokens - (nb - 1) * bt);
        int32_t& dst = S.words[(size_t)S.leaf_tail[k + 1]];
        if (dst != word) {
            dst = word;
            changed.push_back(S.leaf_tail[k + 1]);
            changed.push_back(word);
        }
    }
    return (int32_t)(changed.size() / 2);
}

}  // namespace tp
