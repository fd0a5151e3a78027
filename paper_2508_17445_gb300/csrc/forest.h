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
constexpr int kSchedHeaderWords = 16;
constexpr int32_t kSchedMagic = 0x54505344;
// Units with fewer query rows may run on the CUDA-core path
// (TP_DECODE_CUDA_CORE_SMALL); every other unit runs on tensor cores.
constexpr int kTensorMinRows = 16;
// Query rows per mma.sync unit (4 warps x one 16-row MMA tile each).
constexpr int kTensorRowsPerUnit = 64;
// tcgen05 units (128 rows, MMA M) are opt-in: TP_DECODE_TCGEN05 sends chunks
// of at least kTcMinRows stacked rows per kv head and kTcMinTiles blocks,
// TP_DECODE_ALL_TCGEN05 every unit of more than one 16-row MMA tile. By
// default every unit runs on mma.sync, which measured faster on GB300: the
// tcgen05 pipeline pays a longer start and drain per unit.
constexpr int kTcMinRows = 64;
constexpr int kTcMinTiles = 32;
constexpr int kTcAnyRows = 17;
constexpr int kTcRowsPerUnit = 128;
// Longest unit in pool blocks (the decode kernel keeps a unit's tile words
// in shared memory).
constexpr int kMaxUnitTiles = 128;
// Maximum rows of a CUDA-core unit (two 8-row groups).
constexpr int kCudaCoreMaxRows = 16;
// Pool blocks an append kernel launch can address (larger appends loop).
constexpr int kAppendMaxBlocks = 256;

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
};

struct MergeArgs {
    const int32_t* merge_off;
    const int32_t* merge_slot;
    const float* part_o;
    const float* part_lse;
    uint16_t* out;  // bf16 [n][Hq][hd]
    float* lse;     // [n][Hq], natural log
    int32_t* counters;  // decode's three unit counters, reset to 0 here
    int32_t n;
    int32_t hq;
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
};

// Launchers (kernels.cu). Return cudaSuccess or the launch error.
cudaError_t launch_append(int head_dim, const AppendArgs& a, cudaStream_t s);
// With side != nullptr and both tcgen05 and other units present, the
// tcgen05 units run on `side` concurrently with the rest (fork/join through
// the two events), so a small tcgen05 launch does not leave SMs idle.
cudaError_t launch_decode(int head_dim, const DecodeArgs& a, cudaStream_t s, cudaStream_t side = nullptr,
                          cudaEvent_t fork = nullptr, cudaEvent_t join = nullptr);
cudaError_t launch_merge(int head_dim, const MergeArgs& a, cudaStream_t s);
cudaError_t launch_gather(int head_dim, const GatherArgs& a, int64_t n_tokens, cudaStream_t s);
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
    std::vector<int32_t> words;  // header | units | tiles | occ | merge_off | merge_slot
    int32_t n_units = 0, n_tiles = 0, n_occ = 0, n = 0, n_slots = 0, n_merge = 0, n_tensor = 0, n_tc = 0;
    int64_t off_units = 0, off_tiles = 0, off_occ = 0, off_merge_off = 0, off_merge_slot = 0;
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

    // scheduler scratch (reused across calls)
    std::vector<uint32_t> mark;
    std::vector<int32_t> local;
    uint32_t epoch = 0;

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

    // kernel timing (tp_profile_start / tp_profile_stop)
    bool profiling = false;
    std::vector<cudaEvent_t> ev_pool;
    struct Timed {
        int kind;
        cudaEvent_t a, b;
    };
    std::vector<Timed> timed;
    size_t ev_used = 0;

    // schedule cache: the device copy of the last uploaded schedule
    tp::Schedule sched;
    bool sched_valid = false;
    uint64_t sched_version = 0;
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

   private:
    tp_tree* t_;
    int kind_;
    cudaEvent_t b_ = nullptr;
};

// forest.cpp
tp_status fail(tp_tree* t, tp_status code, const std::string& msg);
tp_status check_live(tp_tree* t, tp_node node, bool need_leaf);
tp_status build_schedule(tp_tree* t, const tp_node* leaves, int32_t n, uint32_t flags, Schedule& out);
void path_tiles(const tp_tree* t, tp_node leaf, std::vector<int32_t>& tiles);
}  // namespace tp
