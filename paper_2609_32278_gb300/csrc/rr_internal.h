// rr_internal.h -- declarations shared by the CUDA translation units of librr.so
// (not part of the public ABI; the public ABI is include/rr.h).
#pragma once
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "rr.h"

namespace rr {

// Tiling of the extend-attention kernel.
constexpr int kBM = 128;          // packed (token, head) rows per Q tile = TMEM lanes
constexpr int kBN = 128;          // keys per KV tile
constexpr int kNQ = 2;            // Q tiles per work unit (two softmax warpgroups ping-pong)
constexpr int kCostBuckets = 4096;  // schedule: counting sort on the number of KV tiles

// Device-side bookkeeping of one call (all pointers into the per-device workspace).
struct SchedArgs {
    const int32_t* prefix;
    const int32_t* suffix;
    // decode: when kv_lens is set, the schedule first writes prefix = kv_lens - 1 and suffix = 1 into
    // the two arrays below (which prefix / suffix then point to) and flags kv_lens < 1
    const int32_t* kv_lens;
    int32_t* prefix_out;
    int32_t* suffix_out;
    int32_t B, Hkv;
    int32_t unit_tokens;   // suffix tokens covered by one work unit (kNQ * kBM / G)
    int64_t T;
    int32_t max_pages, ps;
    int64_t max_units;
    int32_t build_units;   // 0: lengths prefix sums only (append)
    int32_t* cu;           // [B+1] exclusive prefix sum of suffix lens
    int32_t* unit_off;     // [B+1] first work unit of each agent
    int4* units;           // [max_items] (agent, kv head | split << 8 | nsplit << 16, unit, KV tiles of the unit),
                           // most expensive first
    int32_t* item_slot;    // [max_items] partial-result slot of a split item, -1 if the unit is not split
    int4* split_units;     // [units] split units for the combine: (agent, kv head | nsplit << 16, unit, first slot)
    int32_t* n_split;      // number of split units
    int32_t split_grid;    // persistent grid size; 0 disables splitting
    int32_t split_waves;   // a split aims at this many waves of items (2 if 0); slots needed: (waves + 2) x grid
    // decode over a shared prefix (rr_decode_attention_shared): the schedule covers each agent's private keys
    // (kv_lens - lens_offset of them); every unit writes partial results, into slots after `extra_slots`
    // slots reserved for the shared prefix's pieces; unit_slot[b * Hkv + g] receives the unit's first slot.
    // shared_pages > 0: every agent's first shared_pages page-table entries must equal agent 0's.
    int32_t lens_offset;
    int32_t extra_slots;
    int32_t* unit_slot;
    const int32_t* page_table;
    int32_t shared_pages;
    int32_t min_prefix;    // every agent's prefix must be at least this long (extend over a shared prefix)
    int32_t* n_units;      // number of items
    int32_t* lens_ok;
    int32_t* grid_sync;    // set to 0 (the fused extend step's grid-barrier counter), if non-null
    int32_t* err;
};

struct AppendArgs {
    const uint4* k_new;
    const uint4* v_new;
    uint4* k_pool;
    uint4* v_pool;
    const int32_t* page_table;
    const int32_t* prefix;
    const int32_t* suffix;     // read only when the kernel checks the lengths itself (self_lens)
    const int32_t* cu;
    const int32_t* lens_ok;
    int32_t* err;
    int64_t T;
    int64_t num_pages;
    int32_t B, max_pages, ps;
    int32_t row16;         // 16-byte vectors per token row (Hkv * D * 2 / 16)
    // rotary embedding of K (null: plain copy): table [rope_max_pos][D/2] float2 (cos, sin)
    const float2* rope;
    int32_t rope_max_pos;
    int32_t hkv, d16;      // KV heads; D / 16 = rotation pair vectors per head
    // batches of at most kAppendSelfLensMaxB agents: the append kernel checks the lengths and takes the suffix
    // prefix sums itself, in every block, and runs without the schedule kernel in front of it
    int32_t self_lens;
};
constexpr int kAppendSelfLensMaxB = 2047;

struct AttnArgs {
    CUtensorMap tm_q;      // q   [T][Hq][D]        box {64, G, 128/G}, 128B swizzle
    CUtensorMap tm_k;      // k_pool [pages*ps][Hkv*D] box {64, ps},   128B swizzle
    CUtensorMap tm_v;      // v_pool, same
    const int32_t* page_table;
    const int32_t* prefix;
    const int32_t* suffix;
    const int32_t* cu;
    const int4* units;
    const int32_t* n_units;
    const int32_t* item_slot;  // partial-result slot of each item (-1: not split, write out directly)
    float* part_o;         // [slots][kNQ * kBM][D] fp32 unnormalised partial outputs of split items
    float2* part_ml;       // [slots][kNQ * kBM] (running max in log2 units, sum of weights)
    int32_t* err;
    void* out;             // [T][Hq][D] bf16
    int64_t num_pages;
    int32_t Hq, G, ps, max_pages;
    int32_t tq;            // tokens per Q tile = 128 / G
    int32_t oob_row;       // first row past the pool (TMA fills it with zeros)
    float scale_log2;      // softmax scale * log2(e)
    long long wait_limit;  // cycles a pipeline wait may take before the kernel gives up (RR_ERR_TIMEOUT):
                           // every wait of the decode kernel, the extend kernel's stage watcher
    uint32_t wait_hint_ns; // how long one try of such a wait may suspend the thread
    // fused extend step only: the kernel first writes k_new / v_new into the pool (K rotated when rope is
    // set), then crosses a grid barrier on grid_sync (zeroed by the schedule kernel) before the attention
    int32_t* grid_sync;
    const uint4* knew;     // k_new / v_new rows and pool rows, 16-byte vectors
    const uint4* vnew;
    uint4* kpool;
    uint4* vpool;
    int32_t row16;         // 16-byte vectors per token row (Hkv * D * 2 / 16)
    // rotary embedding of q (null: q is used as given): table [rope_max_pos][D/2] float2 (cos, sin)
    const float2* rope;
    int32_t rope_max_pos;
    // decode: partial-result rows per slot (16: one row per query head of a KV head)
    int32_t rows_per_slot;
    // decode over a shared prefix: the private items' page-table columns start at page0; the shared-prefix
    // items (kGroup) each cover `group_agents` consecutive agents of one KV head over a piece of the
    // shared_tiles shared KV tiles, their queries loaded through tm_qg (box {64, G, group_agents})
    int32_t page0;
    const int32_t* unit_slot;  // first partial slot of unit (agent b, KV head g) at b * Hkv + g
    int32_t group_items, group_ns, group_agents, groups_per_head, shared_tiles, batch;
    CUtensorMap tm_qg;
    // extend over a shared prefix (rr_extend_attention_shared): cas_tiles = shared keys / 128; the shared pass
    // runs cas_units implicit units over all cas_T suffix rows; partials [cas_T * Hq][D] and [cas_T * Hq]
    int32_t cas_tiles, cas_units;
    int64_t cas_T;
    float* cas_o;
    float2* cas_ml;
};

struct CombineArgs {
    const int4* split_units;  // (agent, kv head | nsplit << 16, unit, first slot)
    const int32_t* n_split;
    const float* part_o;
    const float2* part_ml;
    const int32_t* suffix;
    const int32_t* cu;
    void* out;
    int32_t Hq, G, D, tq;
    int32_t rows;          // partial rows per slot: kNQ * kBM (extend) or 16 (decode)
};

// Launch `kernel` so that it may start while the kernel before it on the stream finishes (programmatic
// dependent launch: the schedule before the append and attention kernels, the attention kernel before
// the split-K combine); the kernel must call ptx::griddep_wait() before it reads anything the kernels
// before it write.
template <typename... KArgs, typename... Args>
cudaError_t launch_after_sched(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                               Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// The pipeline wait budget the attention kernels get (rr_set_wait_limit; 2^33 cycles, ~4 s at 2 GHz, by default).
long long wait_limit_cycles();

cudaError_t launch_sched(const SchedArgs& a, cudaStream_t st);
cudaError_t launch_combine(const CombineArgs& a, int grid, cudaStream_t st);
cudaError_t launch_kv_append(const AppendArgs& a, int sm_count, cudaStream_t st);
// Returns cudaErrorInvalidValue for an unsupported head dim.  fused: the one-launch extend step (the
// kernel writes k_new / v_new into the pool, waits at a grid barrier on a.grid_sync, then attends over
// the pool; a cooperative launch).  a.rope set: q is rotated in shared memory as each Q tile lands (and,
// fused, each K row on its way into the pool).
cudaError_t launch_extend_attention(const AttnArgs& a, int head_dim, int grid, cudaStream_t st, bool fused = false);
// The two passes of rr_extend_attention_shared (shared_pass: every suffix row against the shared keys, an
// ordinary launch; otherwise the schedule's units over the private keys, merging, as the schedule's dependent).
cudaError_t launch_extend_cascade(const AttnArgs& a, int head_dim, int grid, cudaStream_t st, bool shared_pass);
// Rotary table (rope.cu): table[p][i] = (cos, sin) of p * base^(-2i/D), p < max_pos, i < D/2.
cudaError_t launch_rope_table(float2* out, int max_pos, int head_dim, double base, int sm_count, cudaStream_t st);
size_t extend_attention_smem_bytes(int head_dim);
// Decode: the same arguments (tm_q boxes one token of G heads); units from the schedule run on
// prefix = kv_lens - 1 and suffix = 1, which the schedule writes (SchedArgs::kv_lens).
cudaError_t launch_decode_attention(const AttnArgs& a, int head_dim, int grid, cudaStream_t st);
// The shared-prefix items of rr_decode_attention_shared (a.group_items of them, one KV head x group_agents
// agents x a piece of the shared tiles each); partial results into the agents' first unit slots.
cudaError_t launch_decode_shared_prefix(const AttnArgs& a, int head_dim, int grid, cudaStream_t st);

}  // namespace rr
