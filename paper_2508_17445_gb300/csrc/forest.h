// forest.h -- internal declarations shared by the host code (forest.cpp,
// capi.cpp) and the CUDA launchers (kernels.cu). Not part of the C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/treepo.h"

namespace tp {

// Tile word: one pool block of a path, block << 7 | (valid tokens - 1).
constexpr int kTileValidBits = 7;
constexpr int32_t kMaxPoolBlocks = 1 << 24;
// Unit record: 8 int32 words (layout in treepo.h, tp_debug_schedule).
constexpr int kUnitWords = 8;
enum UnitWord { U_TILE_OFF, U_N_TILES, U_OCC_OFF, U_ROW0, U_N_ROWS, U_SLOT_BASE, U_KVH, U_KIND };
enum UnitKind { KIND_CUDA_CORE = 0, KIND_TENSOR = 1, KIND_TC = 2 };
// Launch flavour of tensor units under a causal mask (prefill schedules; the
// unit words still say KIND_TENSOR).
constexpr int KIND_PREFILL = 3;
constexpr int kSchedHeaderWords = 16;
// Merge record of an occurrence: [slot count, up to 15 slots] (the count is
// -1 when the occurrence has more slots: the merge then reads the CSR).
// Fixed-size, so the merge finds it without reading merge_off first.
constexpr int kMergeRecWords = 16;
constexpr int32_t kSchedMagic = 0x54505344;
// Units with fewer query rows may run on the CUDA-core path
// (TP_DECODE_CUDA_CORE_SMALL); every other unit runs on tensor cores.
constexpr int kTensorMinRows = 16;
// Query rows per mma.sync unit (4 warps x one 16-row MMA tile each).
constexpr int kTensorRowsPerUnit = 64;
// tcgen05 units (128 rows, MMA M): by default every unit of more than one
// 16-row MMA tile (kTcAnyRows); TP_DECODE_TCGEN05 alone keeps tcgen05 to
// chunks of at least kTcMinRows stacked rows per kv head and kTcMinTiles
// blocks; TP_MMA_SYNC runs all stacked rows on mma.sync in 64-row units.
constexpr int kTcMinRows = 64;
constexpr int kTcMinTiles = 32;
constexpr int kTcAnyRows = 17;
constexpr int kTcRowsPerUnit = 128;
// Decode calls reading less K/V than this (about a microsecond of HBM time)
// keep every unit on mma.sync: one attention kernel, no side stream.
constexpr int64_t kSmallCallBytes = 1 << 20;
// Longest unit in pool blocks (the decode kernel keeps a unit's tile words
// in shared memory).
constexpr int kMaxUnitTiles = 128;
// Maximum rows of a CUDA-core unit (two 8-row groups).
constexpr int kCudaCoreMaxRows = 16;
// Pool blocks an append kernel launch can address (larger appends loop).
constexpr int kAppendMaxBlocks = 256;
// Tokens per pool block (the ABI fixes block_tokens to 32).
constexpr int kTileTokens = 32;

// ---- index checks of the bounds-checked build -----------------------------
// Built with -DTP_BOUNDS_CHECK (build.py's checked variant), every kernel
// checks each schedule-derived index before it uses it -- tile words against
// the pool, unit records against the schedule's sections, occurrence entries
// against the rows of Q/O, partial slots, merge ranges, pool slots of token
// appends, schedule patch positions -- and on a failed check sets
// kErrBounds in the device error word and skips the access (no trap). The
// predicates are shared with the host, where tp_debug_check_schedule runs
// them over a schedule without a GPU. In the default build the checks
// compile away.
#if defined(__CUDACC__)
#define TP_HD __host__ __device__ __forceinline__
#else
#define TP_HD inline
#endif
#ifdef TP_BOUNDS_CHECK
constexpr bool kBoundsCheck = true;
#else
constexpr bool kBoundsCheck = false;
#endif
constexpr int32_t kErrBounds = 64;

// Sizes of everything a schedule's words index into.
struct Extents {
    int64_t pool_blocks = 0;  // pool blocks
    int32_t n_tiles = 0;      // tile words
    int32_t n_occ = 0;        // occurrence-list entries
    int32_t n = 0;            // leaf occurrences (query rows of Q, O, LSE)
    int32_t n_slots = 0;      // partial slots
    int32_t n_merge = 0;      // merge entries
    int32_t hkv = 0;
    int32_t group = 1;
};

TP_HD bool in_range(int64_t i, int64_t n) { return i >= 0 && i < n; }

// Tile word block << 7 | (valid - 1): a pool block and 1..32 valid tokens.
TP_HD bool tile_word_ok(int32_t w, int64_t pool_blocks) {
    return w >= 0 && (int64_t)(w >> kTileValidBits) < pool_blocks && (w & ((1 << kTileValidBits) - 1)) < kTileTokens;
}

// Most query rows a unit of each kind holds.
TP_HD int32_t unit_rows_limit(int32_t kind) {
    return kind == KIND_CUDA_CORE ? kCudaCoreMaxRows : kind == KIND_TC ? kTcRowsPerUnit : kTensorRowsPerUnit;
}

// A unit record: its tiles lie inside the tile section (at most
// kMaxUnitTiles), its rows' occurrence entries inside the occurrence list,
// their partial slots below n_slots (slot_base -1: the rows' only unit writes
// O and LSE directly, prefill schedules only), its kv head below hkv.
TP_HD bool unit_ok(int32_t tile_off, int32_t n_tiles, int32_t occ_off, int32_t row0, int32_t n_rows,
                   int32_t slot_base, int32_t kvh, int32_t rows_limit, bool direct_ok, const Extents& x) {
    if (n_tiles < 1 || n_tiles > kMaxUnitTiles || tile_off < 0 || (int64_t)tile_off + n_tiles > x.n_tiles)
        return false;
    if (n_rows < 1 || n_rows > rows_limit || row0 < 0 || occ_off < 0 || kvh < 0 || kvh >= x.hkv || x.group < 1)
        return false;
    const int64_t last = ((int64_t)row0 + n_rows - 1) / x.group;  // the unit's last occurrence group
    if ((int64_t)occ_off + last >= x.n_occ) return false;
    if (slot_base < 0) return direct_ok && slot_base == -1;
    return (int64_t)slot_base + last < x.n_slots;
}

// Occurrence `i`'s merge entries [beg, end).
TP_HD bool merge_range_ok(int32_t beg, int32_t end, int32_t n_merge) { return 0 <= beg && beg <= end && end <= n_merge; }

// ---- device launch arguments --------------------------------------------
struct DecodeArgs {
    const int32_t* units;
    const int32_t* tiles;
    const int32_t* occ;
    const uint16_t* q;  // bf16 [n][Hq][hd]
    const uint8_t* pool;
    float* part_o;      // [slot][Hq][hd], normalised partial output
    float* part_lse;    // [slot][Hq], log2-domain partial LSE
    int32_t* err;
    const int32_t* vis = nullptr;       // prefill: visible path tokens per occurrence (nullptr: decode)
    const int32_t* unit_pos = nullptr;  // prefill: path position of each unit's first token
    uint16_t* out = nullptr;            // units with slot_base < 0 write O (bf16 [n][Hq][hd]) and
    float* out_lse = nullptr;           // LSE (natural log) here directly: their rows have no other part
    int32_t* counters;    // [3] next unit per kind (0 at launch; the merge re-arms them)
    int32_t* counter;     // the counter of the launch in flight (set by the launcher)
    int32_t n_tc_units;      // units [0, n_tc) are tcgen05 units,
    int32_t n_tensor_units;  // then n_tensor mma.sync units, then CUDA-core units
    int32_t unit_begin, unit_end;  // unit range of the launch in flight
    int64_t block_bytes;  // bytes of one pool block (K and V, all kv heads)
    int32_t head_bytes;   // bytes of one (block, K|V, kv head) tile
    int32_t n_units;
    int32_t hq;
    int32_t hkv;
    int32_t group;
    float qk_scale_log2;  // log2(e) / sqrt(hd)
    int32_t kv_read_once = 0;  // decode, default routing: the mma.sync kernel's units, and the tcgen05
                               // units of single-row-block items, read disjoint K/V (copied in as L2
                               // evict-first)
    Extents ext;  // what the schedule indexes into (bounds-checked build)
};

struct MergeArgs {
    const int32_t* merge_off;
    const int32_t* merge_slot;
    const int32_t* merge_rec;  // [n][kMergeRecWords], or null: the CSR only (prefill schedules)
    const float* part_o;
    const float* part_lse;
    uint16_t* out;  // bf16 [n][Hq][hd]
    float* lse;     // [n][Hq], natural log
    int32_t* counters;  // decode's three unit counters, reset to 0 here
    int32_t n;
    int32_t hq;
    int32_t* err = nullptr;  // device error word (bounds-checked build)
    int32_t n_merge = 0;     // merge entries and partial slots (bounds-checked build)
    int32_t n_slots = 0;
};

struct AppendArgs {
    const void* k;
    const void* v;
    uint8_t* pool;
    int64_t block_bytes;
    int32_t head_bytes;
    int32_t hkv;
    int32_t first_row;  // row of the first appended token inside blocks[0]
    int32_t n_tokens;
    int32_t* err = nullptr;      // bounds-checked build: device error word
    int64_t pool_blocks = 0;     // and the pool size the blocks are checked against
    int32_t blocks[kAppendMaxBlocks];
};

struct GatherArgs {
    const int32_t* tiles;
    const uint8_t* pool;
    void* k_out;
    void* v_out;
    int64_t block_bytes;
    int32_t head_bytes;
    int32_t hkv;
    int32_t n_tiles;
    int32_t block_tokens;
    int32_t* err = nullptr;   // bounds-checked build: device error word
    int64_t pool_blocks = 0;  // and the pool size
};

// One token per listed node: row i of k / v goes to pool slot slots[i]
// (block * block_tokens + row).
struct AppendTokensArgs {
    const void* k;
    const void* v;
    const int32_t* slots;
    uint8_t* pool;
    int64_t block_bytes;
    int32_t head_bytes;
    int32_t hkv;
    int32_t n;
    int32_t* err = nullptr;   // bounds-checked build: device error word
    int64_t pool_blocks = 0;  // and the pool size the slots are checked against
};

// Synthetic activations of the stand-in model (splitmix.h): row i is token
// (node, pos) with node = row_node ? row_node[i] : node0 and
// pos = row_node ? pos0 : pos0 + i; each non-null output gets its tag's values.
struct SynthArgs {
    uint16_t* k;  // [rows][kv_width]
    uint16_t* v;  // [rows][kv_width]
    uint16_t* q;  // [rows][q_width]
    const int32_t* row_node;
    uint64_t seed;
    int64_t rows;
    int32_t kv_width;
    int32_t q_width;
    int32_t node0;
    int32_t pos0;
};

// One token step of the rollout's decode loop (rollout_token_step): the
// stand-in activations of each row's new token, K and V written straight
// into the row's pool slot, Q into q; then the decode schedule's patches.
struct StepArgs {
    const int32_t* row_node;  // [n] node of each row
    const int32_t* slots;     // [n] pool slot of each row's new token
    const int32_t* pairs;     // [2 n_pairs]: (schedule word index, new value)
    int32_t* sched;
    uint8_t* pool;
    uint16_t* q;              // [n][q_width]
    uint64_t seed;
    int64_t block_bytes;
    int32_t head_bytes, hkv, q_width, pos, n, n_pairs;
    int32_t* err = nullptr;     // bounds-checked build: device error word,
    int64_t pool_blocks = 0;    // the pool size the slots are checked against
    int64_t sched_words = 0;    // and the schedule length the patches are
};

// Tree advantage (Eq. tree_ae) over a node table; see tp_tree_advantage.
struct AdvantageArgs {
    const int32_t* parent;  // [n_nodes]
    const int32_t* leaf;    // [n_out]
    const float* reward;    // [n_out]
    float* adv;             // [n_out]
    double* stats;          // [4]: accepted outputs, mean, std, error flag
    uint8_t* ws;            // workspace, advantage_ws_bytes(n_nodes, n_out)
    int32_t n_nodes;
    int32_t n_out;
};
int64_t advantage_ws_bytes(int64_t n_nodes, int64_t n_out);

// Launchers (kernels.cu). Return cudaSuccess or the launch error.
cudaError_t launch_append(int head_dim, const AppendArgs& a, cudaStream_t s);
// With side != nullptr and both tcgen05 and other units present, the
// tcgen05 units run on `side` concurrently with the rest (fork/join through
// the two events), so a small tcgen05 launch does not leave SMs idle.
cudaError_t launch_decode(int head_dim, const DecodeArgs& a, cudaStream_t s, cudaStream_t side = nullptr,
                          cudaEvent_t fork = nullptr, cudaEvent_t join = nullptr);
cudaError_t launch_merge(int head_dim, const MergeArgs& a, cudaStream_t s);
cudaError_t launch_gather(int head_dim, const GatherArgs& a, int64_t n_tokens, cudaStream_t s);
// sched[pairs[2k]] = pairs[2k + 1] for k < n (sched_words and err: the
// bounds-checked build's limit and error word).
cudaError_t launch_patch(int32_t* sched, const int32_t* pairs, int32_t n, cudaStream_t s, int64_t sched_words = 0,
                         int32_t* err = nullptr);
cudaError_t launch_wait_probe(int32_t* err, uint64_t limit_ns, cudaStream_t s);
cudaError_t launch_append_tokens(int head_dim, const AppendTokensArgs& a, cudaStream_t s);
cudaError_t launch_synth(const SynthArgs& a, cudaStream_t s);
cudaError_t launch_rollout_step(int head_dim, const StepArgs& a, cudaStream_t s);
cudaError_t launch_advantage(const AdvantageArgs& a, cudaStream_t s);
int decode_smem_bytes(int head_dim);
// Device address of the library's static scratch array (tp_decode_noalloc).
cudaError_t noalloc_scratch(void** device_ptr);

// ---- host objects ---------------------------------------------------------
struct Node {
    int32_t parent = -1;
    int32_t state = 0;  // 0 leaf, 1 frozen, 2 dead
    int32_t n_tokens = 0;
    int32_t kids_live = 0;
    int64_t path_before = 0;  // tokens on the path above this node
    std::vector<int32_t> blocks;
};

// Lowest-index-first block allocator over a bitmap.
class BlockPool {
   public:
    void init(int64_t n_blocks);
    int64_t free_count() const { return free_; }
    int64_t size() const { return n_; }
    // Appends `count` blocks to `out`, lowest free first; false if short.
    bool alloc(int64_t count, std::vector<int32_t>& out);
    void release(const std::vector<int32_t>& blocks);

   private:
    std::vector<uint64_t> bits_;  // 1 = free
    int64_t n_ = 0, free_ = 0, hint_ = 0;
};

struct Schedule {
    // header | units | tiles | occ | merge_off | merge_slot, then for a
    // decode schedule merge_rec [n][16], for a prefill one unit_pos
    // [n_units] | vis [n]
    std::vector<int32_t> words;
    int32_t n_units = 0, n_tiles = 0, n_occ = 0, n = 0, n_slots = 0, n_merge = 0, n_tensor = 0, n_tc = 0;
    int64_t off_units = 0, off_tiles = 0, off_occ = 0, off_merge_off = 0, off_merge_slot = 0;
    bool prefill = false;
    bool kv_read_once = false;  // see DecodeArgs::kv_read_once
    int64_t off_unit_pos = 0, off_vis = 0, off_merge_rec = 0;
    // (leaf node, word index of the last tile of that leaf) for every place a
    // listed leaf's last block appears: appends that stay inside that block
    // change only these words (see patch_schedule)
    std::vector<int32_t> leaf_tail;
};

// A run of path blocks read with one stacked row set (a node, or a chain of
// nodes with the same occurrence set).
struct Item {
    int32_t occ_off;  // into the occurrence list
    int32_t n_occ;
    int32_t tile_off;  // into the tile list
    int32_t n_tiles;
};

// Scheduler scratch kept by the tree so repeated schedules reuse their
// buffers instead of allocating (and page-faulting) fresh ones per call.
struct SchedScratch {
    std::vector<uint32_t> mark;   // per node id: epoch of the last visit
    std::vector<int32_t> local;   // per node id: index among the touched nodes
    uint32_t epoch = 0;
    std::vector<int32_t> touched, cnt, start, fill, all_occ, order, item_of, item_cnt, item_start, item_nodes;
    std::vector<Item> items;
    std::vector<int32_t> occ, tiles, tail_node, tail_tile;
    std::vector<int32_t> units[3], sorted, bucket;
    std::vector<int32_t> pair_occ, pair_slot, merge_off, merge_pos, merge_slot;
    std::vector<int32_t> tile_pos, node_tile_off, vis;  // prefill
    std::vector<int32_t> step_words;                    // rollout_token_step's upload
};

}  // namespace tp

struct tp_tree {
    tp_config cfg{};
    cudaStream_t stream = nullptr;
    std::string err;
    std::vector<tp::Node> nodes;
    tp::BlockPool pool;
    int64_t live_nodes = 0;
    uint64_t version = 0;  // bumped on every structural change

    uint64_t struct_version = 0;  // bumped on changes other than appends inside a node's last block

    // scheduler scratch (reused across calls)
    tp::SchedScratch scratch;

    // device scratch owned by the library
    int32_t* d_err = nullptr;  // [0] device error flag, [1..3] decode unit counters
    int32_t* d_sched = nullptr;
    int64_t d_sched_cap = 0;  // words
    float* d_part = nullptr;  // partial o then partial lse
    int64_t d_part_cap = 0;   // floats
    int32_t* h_pinned[2] = {nullptr, nullptr};
    int64_t h_pinned_cap[2] = {0, 0};
    cudaEvent_t h_pinned_ev[2] = {nullptr, nullptr};
    int pinned_next = 0;
    int32_t* d_gather_tiles = nullptr;
    int64_t d_gather_cap = 0;
    cudaStream_t side = nullptr;  // second stream for concurrent tcgen05 units
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;

    // prefill schedules (rebuilt every call): two device buffers used in
    // turn, uploaded on a copy stream of their own once the kernels that read
    // the buffer two calls back are done, so a call's upload overlaps the
    // previous call's attention; a host Schedule of their own (the decode
    // cache keeps its own)
    tp::Schedule pf_sched;
    cudaStream_t pf_copy = nullptr;
    int32_t* d_pf[2] = {nullptr, nullptr};
    int64_t d_pf_cap[2] = {0, 0};  // words
    int32_t* h_pf[2] = {nullptr, nullptr};
    int64_t h_pf_cap[2] = {0, 0};  // words
    cudaEvent_t pf_up[2] = {nullptr, nullptr};    // buffer's upload landed
    cudaEvent_t pf_done[2] = {nullptr, nullptr};  // kernels reading the buffer finished
    uint64_t pf_calls = 0;

    // host-buffer calls (tp_decode_host, tp_prefill_host): two staging slots
    // used in turn, uploads and downloads on streams of their own so that a
    // call's copies overlap its neighbours' attention
    cudaStream_t hp_h2d = nullptr, hp_d2h = nullptr;
    cudaEvent_t hp_up[2] = {nullptr, nullptr};    // slot's Q uploaded
    cudaEvent_t hp_done[2] = {nullptr, nullptr};  // slot's attention finished
    cudaEvent_t hp_down[2] = {nullptr, nullptr};  // slot's O and LSE downloaded
    void* hp_q[2] = {nullptr, nullptr};
    void* hp_o[2] = {nullptr, nullptr};
    void* hp_lse[2] = {nullptr, nullptr};
    int64_t hp_q_cap[2] = {0, 0}, hp_o_cap[2] = {0, 0}, hp_lse_cap[2] = {0, 0};  // bytes
    uint64_t hp_calls = 0;

    // kernel timing (tp_profile_start / tp_profile_stop)
    bool profiling = false;
    std::vector<cudaEvent_t> ev_pool;
    struct Timed {
        int kind;
        cudaEvent_t a, b;
        int kernels;  // kernels launched inside the bracket
    };
    std::vector<Timed> timed;
    size_t ev_used = 0;
    int64_t untimed[4] = {0, 0, 0, 0};  // kernels counted without their own events, per kind

    // schedule cache: the device copy of the last uploaded schedule
    tp::Schedule sched;
    bool sched_valid = false;
    uint64_t sched_version = 0;
    uint64_t sched_struct = 0;  // struct_version the cached schedule was built at
    std::vector<int32_t> patch_words;
    int32_t* d_patch = nullptr;
    int64_t d_patch_cap = 0;

    // tp_append_tokens: pool slot of each appended token
    std::vector<int32_t> tok_slots;
    int32_t* d_tok_slots = nullptr;
    int64_t d_tok_slots_cap = 0;
    uint32_t sched_flags = 0;
    std::vector<int32_t> sched_leaves;
};

namespace tp {
enum KernelKind { KK_DECODE = 0, KK_MERGE = 1, KK_APPEND = 2, KK_GATHER = 3 };
// Brackets one launch with timing events while profiling is on.
class LaunchTimer {
   public:
    LaunchTimer(tp_tree* t, int kind);
    ~LaunchTimer();
    void kernels(int n);  // the bracket launched n kernels (default 1)

   private:
    tp_tree* t_;
    int kind_;
    cudaEvent_t b_ = nullptr;
    size_t index_ = 0;
};
// Counts n kernels of a kind while profiling, without timing them.
void count_kernels(tp_tree* t, int kind, int n);

// capi.cpp
tp_status cuda_fail(tp_tree* t, cudaError_t e, const char* what);
// Grow a device buffer to at least `need` bytes (contents are not kept);
// waits for the tree's stream first so no queued kernel still reads it.
tp_status ensure_device_bytes(tp_tree* t, void** ptr, int64_t* cap, int64_t need, const char* what);
// Copy `words` int32 words to device `dst` on the tree's stream through a
// double-buffered pinned staging area; a staging buffer is reused only after
// its previous copy has completed.
tp_status stage_upload(tp_tree* t, int32_t* dst, const int32_t* src, int64_t words);
tp_status append_tokens_plan(tp_tree* t, const tp_node* nodes, int32_t n, int64_t* need);
void append_tokens_unplan(tp_tree* t, const tp_node* nodes, int32_t n);
void append_tokens_commit(tp_tree* t, const tp_node* nodes, int32_t n, int64_t need);
tp_status rollout_token_step(tp_tree* t, const tp_node* nodes, int32_t n, int32_t* d_buf, int64_t buf_words,
                             uint64_t seed, int32_t pos, uint16_t* q, uint32_t decode_flags);

// forest.cpp
tp_status fail(tp_tree* t, tp_status code, const std::string& msg);
tp_status check_live(tp_tree* t, tp_node node, bool need_leaf);
tp_status build_schedule(tp_tree* t, const tp_node* leaves, int32_t n, uint32_t flags, Schedule& out);
// Prefill: the last m[i] tokens of nodes[i] attend causally to their root-
// to-node path. Occurrence q (query token, packed node by node) sees the
// path's first vis[q] tokens; its rows are kept per node in blocks of whole
// GQA groups, and each block reads the node's path tiles up to its last
// visible token, in chunks of at most kMaxUnitTiles tiles.
tp_status build_prefill_schedule(tp_tree* t, const tp_node* nodes, const int32_t* m, int32_t n, uint32_t flags,
                                 Schedule& out);
// Refresh the last-tile words of S's leaves from the tree (valid after
// appends that stayed inside those leaves' last blocks); `changed` receives
// (word index, new word) pairs. Returns the number of changed words.
int32_t patch_schedule(const tp_tree* t, Schedule& S, std::vector<int32_t>& changed);
void path_tiles(const tp_tree* t, tp_node leaf, std::vector<int32_t>& tiles);
}  // namespace tp
