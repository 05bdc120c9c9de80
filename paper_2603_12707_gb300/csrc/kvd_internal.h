// Internal declarations shared by the host library (kvd_host.cpp) and the
// kernel translation units.  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvd {

constexpr int kPageSize = 16;          // tokens per page (the only supported P)
constexpr int kMaxGroup = 8;           // query heads per KV head handled by one MMA N-tile
constexpr int kMaxChunks = 64;         // work items per (row, KV head) at most
constexpr int kChunkCap = 32;          // the usual cap; 64 only when few rows must fill the GPU
constexpr int kChunkCapGqa = 16;       // GQA: the merge variant for 16 items fits beside the split pass
constexpr int kMaxItemPages = 1024;    // largest target item size a caller may request
constexpr int kPatchMax = 1024;        // step entries carried in one launch's parameters
constexpr int kScatterMax = 2048;      // int32 updates carried in one launch's parameters
constexpr int kVarlenMax = 512;        // token blocks carried in one bulk-write launch's parameters

// One work item of a step's split plan: consecutive pages [first_page,
// first_page + n_pages) of batch row b.  Items are expanded over the H_kv
// heads at launch time: item = entry * H_kv + g.
struct PlanEntry {
    int32_t b;          // batch row (q / out row)
    int32_t seq;        // sequence id (page-table row)
    int32_t len;        // tokens attended, including this step's token
    int32_t first_page; // first logical page of the item
    int32_t n_pages;    // pages of the item (>= 1)
    int32_t chunk;      // index of the item among the row's items
    int32_t n_chunks;   // items of the row
    int32_t slot_base;  // first partial slot of the row; slot = (slot_base + chunk) * H_kv + g
};

// Target item size of the row planned at position i of n (rows are planned
// longest first): the last rows get smaller items, so a launch ends on short
// items and the warps run out of work at nearly the same time.
__host__ __device__ inline int row_item_pages(int T, int i, int n)
{
    if (100 * (int64_t)i >= 95 * (int64_t)n) return T >= 8 ? T / 8 : 1;
    if (100 * (int64_t)i >= 85 * (int64_t)n) return T >= 4 ? T / 4 : 1;
    if (10 * (int64_t)i >= 7 * (int64_t)n) return T >= 2 ? T / 2 : 1;
    return T;
}

// Split policy shared by host and device.  A row of np pages is cut into
// nch items of near-equal size: the target size T, raised for long rows so a
// row never has more than `cap` items (which bounds the merge).
__host__ __device__ inline int row_chunks(int np, int T, int cap = kChunkCap)
{
    const int t_row = (np + cap - 1) / cap;
    const int Tb = T > t_row ? T : t_row;
    return (np + Tb - 1) / Tb;
}

// Pages [first, first + n) of item c of nch over np pages.
__host__ __device__ inline void chunk_range(int np, int nch, int c, int* first, int* n)
{
    const int base = np / nch, extra = np % nch;
    *first = c * base + (c < extra ? c : extra);
    *n = base + (c < extra ? 1 : 0);
}

// Per-step update, passed by value in kernel parameters.
struct StepPatch {
    int32_t n;                     // entries in this launch
    int32_t b0;                    // batch row of entry 0
    int32_t seq[kPatchMax];
    int32_t new_len[kPatchMax];
    int32_t new_page[kPatchMax];   // page taken for position new_len-1, or -1
};

struct PlanArgs {
    int32_t build;       // build the plan in this launch (last launch of a step)
    int32_t batch;
    int32_t item_pages;  // target pages per work item (T)
    int32_t max_pages;   // page-table row length
    int32_t use_order;   // rows are planned in order[] (else batch order)
    int32_t order[kPatchMax];
    int32_t* step_seq;   // [max_seqs] batch row -> sequence id
    int32_t* seq_len;    // [max_seqs]
    int32_t* page_table; // [max_seqs][max_pages]
    PlanEntry* plan;     // [n_entries]
    int2* rows;          // [batch]: (first partial slot, items) of each batch row
    int32_t chunk_cap;   // items per row at most (kChunkCap or kMaxChunks)
    int32_t* page_ids;   // [entries][page_stride]: page ids of each entry's pages
    int32_t page_stride;
    int32_t* err;
    uint32_t* step_no;   // step counter, advanced by the launch that builds the plan
};

// kv_begin_step_device: the step's lazy allocation and plan, on the device.
struct StepDevArgs {
    int32_t batch;
    int32_t max_seqs;         // sequence ids outside [0, max_seqs) fail their row
    int32_t item_pages;       // target pages per work item (T)
    int32_t max_pages;        // page-table row length
    int32_t max_entries;      // capacity of plan
    const int32_t* seq_ids;   // [batch] sequence ids (device)
    int32_t* free_pages;      // device free stack; the next page is free_pages[*free_top - 1]
    int32_t* free_top;
    int32_t* step_seq;        // out: [batch] sequence of each row, -1 where the row's step failed
    int32_t* seq_len;
    int32_t* page_table;
    PlanEntry* plan;
    int2* rows;
    int32_t* n_entries;       // out: plan entries of the step
    int32_t chunk_cap;        // items per row at most (kChunkCap or kMaxChunks)
    int32_t* page_ids;        // [max_entries][page_stride]: page ids of each entry's pages
    int32_t page_stride;
    int32_t* err;
    uint32_t* step_no;        // step counter, advanced once per step
};

struct ScatterI32 {
    int32_t n;
    int32_t idx[kScatterMax];
    int32_t val[kScatterMax];
};

// Sequence reservation or release on the device free stack (device-side
// steps enabled): the same pages, in the same order, as the host allocator.
struct SeqOpArgs {
    int32_t free_seq;         // 0: reserve n tokens, 1: release every page of the sequence
    int32_t seq, n;
    int32_t max_pages;        // page-table row length
    int32_t* free_pages;      // device free stack; the next page is free_pages[*free_top - 1]
    int32_t* free_top;
    int32_t* seq_len;
    int32_t* page_table;
    int32_t* err;
};

struct TokenCopyArgs {
    uint16_t* pool_k;         // layer pool base [num_pages][H_kv][P][D]
    uint16_t* pool_v;
    const int32_t* pt_row;    // page-table row of the sequence (device)
    const int32_t* len;       // the sequence's length (device), or null: positions checked on the host
    int64_t num_pages;
    int32_t H_kv, D;
    int32_t first_pos, n;
    uint16_t* tok_k;          // [n][H_kv][D] logical order
    uint16_t* tok_v;
    int32_t to_pool;          // 1: tokens -> pool, 0: pool -> tokens
    int32_t* err;
};

// Bulk write of packed variable-length token blocks into the pools (prefill
// or the vision-prefix handoff).  A tile is the part of one block's position
// range that falls in one page; CTA (x, y) writes tile x of layer
// layer_first + y.
struct VarlenWriteArgs {
    uint16_t* pool_k;            // pool of the first layer written, [num_pages][H_kv][P][D]
    uint16_t* pool_v;
    int64_t pool_layer_stride;   // elements between consecutive layer pools
    const uint16_t* k;           // [n_layers][rows][H_kv][D]
    const uint16_t* v;
    int64_t src_layer_stride;    // rows * H_kv * D
    const int32_t* page_table;   // [max_seqs][max_pages]
    const int32_t* seq_len;      // [max_seqs] (device), or null: positions checked on the host
    int64_t num_pages;
    int32_t max_pages;
    int32_t H_kv, D;
    int32_t n_blocks, n_tiles;
    int32_t* err;
    int32_t tile_start[kVarlenMax + 1];  // first tile of block i; tile_start[n_blocks] = n_tiles
    int32_t seq[kVarlenMax];
    int32_t first_pos[kVarlenMax];
    int32_t n_tok[kVarlenMax];
    int32_t src_row[kVarlenMax];         // packed row of block i's first token
};

struct AppendArgs {
    uint16_t* pool_k;
    uint16_t* pool_v;
    const uint16_t* k_new;    // [B][H_kv][D]
    const uint16_t* v_new;
    const int32_t* step_seq;
    const int32_t* seq_len;
    const int32_t* page_table;
    int64_t num_pages;
    int32_t batch, H_kv, D, max_pages;
    int32_t* err;
};

struct DecodeParams {
    const uint16_t* q;        // [B][H_q][D] bf16
    uint16_t* out;            // [B][H_q][D] bf16
    const int32_t* page_table;
    const PlanEntry* plan;
    float* part_o;            // [slots][G][D]
    float2* part_ml;          // [slots][G]  (running max in log2 units, sum)
    const int2* rows;         // [batch]: (first partial slot, items) per batch row
    const int32_t* item_pages;// [entries][page_stride]: page ids of each plan entry's pages
    int32_t page_stride;
    const int32_t* n_entries_dev; // device-built plan: entries live here (n_items is then a bound)
    int32_t batch;
    uint32_t* queue;          // next item to hand out (zero at launch)
    uint32_t* queue_next;     // the next launch's counter, reset by this one (null: none)
    int32_t* err;
    int64_t num_pages;
    int32_t n_items;
    int32_t H_kv, H_q, G, max_pages;
    float scale_log2;         // softmax scale * log2(e)
    // Fused append (decode_attention_append only): the step's new K/V rows,
    // written into slot len-1 of each row's last page and used in place of
    // what the page held there.
    const uint16_t* k_new;    // [B][H_kv][D] bf16
    const uint16_t* v_new;
    uint16_t* pool_k;         // this layer's pools [num_pages][H_kv][P][D]
    uint16_t* pool_v;
    // 1: the first tensor map covers K and V (one 4-D load per page); 0: two
    // 3-D maps, K and V.
    int32_t kv_map;
    // Early start of a chained launch: the merge pass of each launch writes
    // step * 65536 + tag into every SM's word of start_flags (one word per
    // 128-byte line) once its dependency wait has returned, i.e. once that
    // launch's split pass is complete; a launch with prev_tag != 0 (chained
    // after a launch that has a merge pass) waits for its predecessor's value
    // before its own dependency wait and then brings more of its first item
    // into L2.  step_no is the device step counter (the step kernels count).
    uint32_t* start_flags;
    const uint32_t* step_no;
    uint32_t tag, prev_tag;
    int32_t num_sms;
};

// TMA view of a (page, head) tile: box {64 columns, 16 rows, D/64 column
// halves} of a pool whose rows are D bf16 (row index (page*H_kv + head)*16 +
// slot), 128-byte swizzle; with v_stride_bytes > 0 a fourth dimension of 2
// steps from the K pool to the V pool.  Shared-memory image: [K, V][half]
// [16 rows][128 B].  `encode` is cuTensorMapEncodeTiled.
CUresult encode_tile_map(void* encode_fn, CUtensorMap* map, void* k_pool, int64_t rows, int D,
                         int64_t v_stride_bytes);

// Message returned by kv_last_error() on the calling thread.
void set_last_error(const char* msg);

// ---- launchers (return cudaGetLastError() of the launch) -----------------
cudaError_t launch_scatter_i32(int32_t* base, const ScatterI32& s, cudaStream_t st);
cudaError_t launch_step(const StepPatch& patch, const PlanArgs& plan, cudaStream_t st);
cudaError_t launch_token_copy(const TokenCopyArgs& a, cudaStream_t st);
cudaError_t launch_varlen_write(const VarlenWriteArgs& a, int n_layers, cudaStream_t st);
// Copy each plan entry's page ids from the page table into item_pages
// ([entries][stride]), so the decode kernel reads them alongside the entry.
// entries_dev (if non-null) holds the entry count; `entries` is then its bound.
cudaError_t launch_gather_pages(const PlanEntry* plan, int32_t entries, const int32_t* entries_dev,
                                const int32_t* page_table, int32_t max_pages, int32_t* item_pages, int32_t stride,
                                int num_sms, cudaStream_t st);
cudaError_t launch_step_device(const StepDevArgs& a, cudaStream_t st);
cudaError_t launch_seq_op(const SeqOpArgs& a, cudaStream_t st);
cudaError_t launch_append(const AppendArgs& a, cudaStream_t st);
cudaError_t launch_wait_timeout_check(uint64_t limit_ns, int32_t* status, cudaStream_t st);

// Decode attention: variant chosen by (D, G == 1).
struct DecodeVariant {
    int warps;        // warps per CTA
    int smem_bytes;   // dynamic shared memory per CTA
    int ctas_per_sm;  // occupancy at that shared memory
    int regs;         // registers per thread (the larger of the two variants)
};

// Registers one warp is allocated for `regs` registers per thread (per-thread
// counts are allocated in multiples of 8).
inline int warp_register_allocation(int regs) { return ((regs + 7) / 8) * 8 * 32; }
constexpr int kRegistersPerSubpartition = 16384;   // an SM's 64 K registers over its 4 schedulers
cudaError_t decode_variant_info(int D, bool gqa, DecodeVariant* v);
// Second pass: log-sum-exp merge of the partials of every split row, one warp
// per (row, query head).  pdl: launched with programmatic dependent launch
// (it lets the next kernel start at once and waits for the split pass).
// max_chunks: an upper bound on the items of any row of the step (<= kMaxChunks).
// split_regs_per_subpartition: registers the resident split pass holds on
// each of an SM's four schedulers (0: nothing resident beside it).
cudaError_t launch_merge(int D, bool pdl, int max_chunks, int num_sms, int split_regs_per_subpartition,
                         const DecodeParams& p, cudaStream_t st);
// fused: the append + attention kernel, launched with programmatic dependent
// launch (it streams its first pages before the previous kernel finishes and
// reads q / k_new / v_new and writes anything only after it has).
cudaError_t launch_decode(int D, bool gqa, bool fused, bool pdl, int grid, const CUtensorMap& tk, const CUtensorMap& tv,
                          const DecodeParams& p, cudaStream_t st);

}  // namespace kvd
