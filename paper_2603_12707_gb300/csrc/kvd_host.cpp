// Host side of libkvdecode.so: the C ABI, argument checking, the lazy page
// allocator with its host mirror of the page table, the per-step split plan
// sizing, TMA descriptors, and kernel launches.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "kvd_internal.h"
#include "kvdecode.h"

using namespace kvd;

namespace {

thread_local std::string g_last_error;

int fail(int code, const std::string& msg)
{
    g_last_error = msg;
    return code;
}

#define KVD_CUDA(call)                                                                       \
    do {                                                                                     \
        cudaError_t e_ = (call);                                                             \
        if (e_ != cudaSuccess)                                                               \
            return fail(e_ == cudaErrorMemoryAllocation ? KVC_ERR_OOM : KVC_ERR_CUDA,        \
                        std::string(#call) + ": " + cudaGetErrorString(e_));                 \
    } while (0)

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

void kvd::set_last_error(const char* msg) { g_last_error = msg; }

CUresult kvd::encode_tile_map(void* encode_fn, CUtensorMap* map, void* k_pool, int64_t rows, int D,
                              int64_t v_stride_bytes)
{
    auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(encode_fn);
    // dims (innermost first): 64 columns, rows, D/64 column blocks, [K, V]
    cuuint64_t gdim[4] = {64, (cuuint64_t)rows, (cuuint64_t)(D / 64), 2};
    cuuint64_t gstride[3] = {(cuuint64_t)D * sizeof(uint16_t), 128, (cuuint64_t)v_stride_bytes};
    cuuint32_t box[4] = {64, (cuuint32_t)kPageSize, (cuuint32_t)(D / 64), 2};
    cuuint32_t estride[4] = {1, 1, 1, 1};
    const cuuint32_t rank = v_stride_bytes > 0 ? 4 : 3;
    return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, k_pool, gdim, gstride, box, estride,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

struct kv_cache {
    kvc_config cfg{};
    bool host_only = false;
    int device = 0;
    int group = 1;
    int num_sms = 0;
    DecodeVariant variant{};

    // host allocator state
    std::vector<int32_t> free_stack;            // back() is handed out next
    std::vector<int32_t> lens;                  // -1: sequence id not in use
    std::vector<std::vector<int32_t>> pages;    // logical page -> physical page
    int64_t pages_in_use = 0;
    int32_t live = 0;
    std::vector<uint32_t> stamp;                // duplicate check in kv_begin_step
    uint32_t stamp_gen = 0;

    // device memory
    uint16_t* pools = nullptr;                  // [2][L][num_pages][H_kv][P][D]
    size_t layer_elems = 0;
    int32_t* meta = nullptr;                    // page table [max_seqs][max_pages], then seq_len [max_seqs]
    int32_t* step_seq = nullptr;
    int2* rows = nullptr;                       // per batch row: (first partial slot, items)
    uint32_t* queue = nullptr;                  // two work counters, used by alternate attention launches
    uint32_t* start_flags = nullptr;            // [num_sms][32]: merge passes announce their split pass's end
    uint32_t* step_no = nullptr;                // device step counter
    uint32_t attn_tag = 0;                      // tag of the step's latest attention launch (0: none yet)
    bool prev_merge = false;                    // that launch has a merge pass
    unsigned long long prev_capture = 0;        // its stream-capture sequence (0: not captured)
    uint32_t attn_launches = 0;                 // attention launches so far (selects the counter)
    int64_t launches = 0;                       // kernels launched (reported by kv_cache_query)
    // A fused launch may depend programmatically on the launch before it only
    // if that was an attention launch on the same stream: its early reads
    // (plan, page lists, cached pages) must not race any other writer.
    int64_t chain_launches = -1;                // `launches` right after the last attention launch
    void* chain_stream = nullptr;
    int32_t* err = nullptr;
    PlanEntry* plan = nullptr;
    int64_t plan_cap = 0;
    int32_t* item_pages = nullptr;              // [entries][page_stride]
    int64_t item_pages_cap = 0;
    int32_t page_stride = 0;
    float* part_o = nullptr;
    float2* part_ml = nullptr;
    int64_t slot_cap = 0;
    std::vector<CUtensorMap> tmaps;             // [L]: K and V of a layer

    // device-side steps (kv_begin_step_device): free stack on the device
    bool dev_mode = false;                      // kv_cache_device_steps enabled
    bool dev_dirty = false;                     // the device state moved past the host mirror
    cudaStream_t last_stream = nullptr;         // stream of the cache's latest enqueued work
    cudaStream_t copy_stream = nullptr;         // the cache's own stream for reading its state back
    int32_t dev_max_batch = 0;
    int32_t dev_item_pages = 0;
    int32_t dev_entries_cap = 0;
    int32_t dev_stride = 0;
    int32_t dev_chunk_cap = kChunkCap;
    int32_t* d_free = nullptr;                  // [num_pages]
    int32_t* d_small = nullptr;                 // [0] free top, [1] plan entries of the step

    // current step
    bool step_active = false;
    bool step_dev = false;                      // the step's plan was built on the device
    bool step_split = false;                    // some row of the step has several items
    int32_t step_max_chunks = kMaxChunks;       // bound on the items of a row of the step
    int32_t step_batch = 0;
    int32_t step_entries = 0;
    int32_t split_override = 0;

    int32_t* page_table() const { return meta; }
    int32_t* seq_len_dev() const { return meta + (int64_t)cfg.max_seqs * cfg.max_pages_per_seq; }
    int32_t seq_len_index(int32_t seq) const { return cfg.max_seqs * cfg.max_pages_per_seq + seq; }
    uint16_t* k_pool(int layer) const { return pools + (size_t)layer * layer_elems; }
    uint16_t* v_pool(int layer) const { return pools + ((size_t)cfg.num_layers + layer) * layer_elems; }

    int32_t pop_page()
    {
        const int32_t p = free_stack.back();
        free_stack.pop_back();
        ++pages_in_use;
        return p;
    }
};

namespace {

int check_seq(const kv_cache* c, int32_t seq)
{
    if (seq < 0 || seq >= c->cfg.max_seqs || c->lens[seq] < 0)
        return fail(KVC_ERR_INVALID, "sequence id " + std::to_string(seq) + " is not live");
    return KVC_OK;
}

int check_device(const kv_cache* c, const char* what)
{
    if (c->host_only) return fail(KVC_ERR_INVALID, std::string(what) + ": cache was created host-only");
    return KVC_OK;
}

// Enqueue int32 updates of the page table / lengths.
int push_updates(kv_cache* c, const std::vector<int32_t>& idx, const std::vector<int32_t>& val,
                 cudaStream_t st)
{
    if (c->host_only || idx.empty()) return KVC_OK;
    c->last_stream = st;
    ScatterI32 s;
    for (size_t off = 0; off < idx.size(); off += kScatterMax) {
        const size_t n = std::min<size_t>(kScatterMax, idx.size() - off);
        s.n = (int32_t)n;
        std::memcpy(s.idx, idx.data() + off, n * sizeof(int32_t));
        std::memcpy(s.val, val.data() + off, n * sizeof(int32_t));
        KVD_CUDA(launch_scatter_i32(c->meta, s, st));
        ++c->launches;
    }
    return KVC_OK;
}

int32_t auto_item_pages(const kv_cache* c, int64_t total_units)
{
    // About three work items per resident warp keeps the tail of the
    // persistent schedule short; a GQA item leaves a partial for each of its
    // G query heads, so GQA aims at two.  Items stay within [2, 128] pages
    // (long rows get larger items through the per-row cap on items).
    const int64_t warps = (int64_t)std::max(1, c->num_sms) * std::max(1, c->variant.ctas_per_sm) *
                          std::max(1, c->variant.warps);
    const int64_t per_warp = c->group > 1 ? 2 : 3;
    const int64_t T = (total_units + per_warp * warps - 1) / (per_warp * warps);
    return (int32_t)std::min<int64_t>(128, std::max<int64_t>(2, T));
}

// Items per row at most: twice the usual cap when rows x KV heads x the
// usual cap would leave resident warps without an item and some row (of up
// to max_pages pages) is long enough to use more items of T pages.
// Otherwise 32 for MHA and 16 for GQA: a GQA row of at most 16 items merges
// in one round trip with the 16-item variant, the largest whose registers
// fit beside the resident GQA split pass (Qwen shape: 0.742 at 32, 0.769 at
// 16, 0.756 at 24, 0.686 at 12).
int32_t chunk_cap(const kv_cache* c, int64_t rows, int64_t max_pages, int32_t T)
{
    const int64_t warps = (int64_t)std::max(1, c->num_sms) * std::max(1, c->variant.ctas_per_sm) *
                          std::max(1, c->variant.warps);
    const bool few_units = rows * c->cfg.num_kv_heads * kChunkCap < warps;
    if (few_units && max_pages > (int64_t)kChunkCap * T) return kMaxChunks;
    return c->group > 1 ? kChunkCapGqa : kChunkCap;
}

int grow_scratch(kv_cache* c, int64_t entries, int64_t slots, int64_t page_ids, cudaStream_t st)
{
    // While device steps are enabled, captured graphs may hold these buffers'
    // addresses: they must not move.
    if (c->dev_mode && (page_ids > c->item_pages_cap || entries > c->plan_cap || slots > c->slot_cap))
        return fail(KVC_ERR_INVALID,
                    "the step needs larger plan buffers than kv_cache_device_steps reserved, and graphs "
                    "captured since may use them: disable device steps first");
    if (page_ids > c->item_pages_cap) {
        const int64_t cap = std::max<int64_t>(page_ids, c->item_pages_cap + c->item_pages_cap / 2);
        if (c->item_pages) KVD_CUDA(cudaFreeAsync(c->item_pages, st));
        c->item_pages = nullptr;
        c->item_pages_cap = 0;
        KVD_CUDA(cudaMallocAsync((void**)&c->item_pages, (size_t)cap * sizeof(int32_t), st));
        c->item_pages_cap = cap;
    }
    if (entries > c->plan_cap) {
        const int64_t cap = std::max<int64_t>(entries, c->plan_cap + c->plan_cap / 2);
        if (c->plan) KVD_CUDA(cudaFreeAsync(c->plan, st));
        c->plan = nullptr;
        c->plan_cap = 0;
        KVD_CUDA(cudaMallocAsync((void**)&c->plan, (size_t)cap * sizeof(PlanEntry), st));
        c->plan_cap = cap;
    }
    if (slots > c->slot_cap) {
        const int64_t cap = std::max<int64_t>(slots, c->slot_cap + c->slot_cap / 2);
        if (c->part_o) KVD_CUDA(cudaFreeAsync(c->part_o, st));
        if (c->part_ml) KVD_CUDA(cudaFreeAsync(c->part_ml, st));
        c->part_o = nullptr;
        c->part_ml = nullptr;
        c->slot_cap = 0;
        const size_t G = (size_t)c->group, D = (size_t)c->cfg.head_dim;
        KVD_CUDA(cudaMallocAsync((void**)&c->part_o, (size_t)cap * G * D * sizeof(float), st));
        KVD_CUDA(cudaMallocAsync((void**)&c->part_ml, (size_t)cap * G * sizeof(float2), st));
        c->slot_cap = cap;
    }
    return KVC_OK;
}

void release_device(kv_cache* c)
{
    if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
    cudaFree(c->pools);
    cudaFree(c->meta);
    cudaFree(c->step_seq);
    cudaFree(c->rows);
    cudaFree(c->queue);
    cudaFree(c->start_flags);
    cudaFree(c->step_no);
    cudaFree(c->err);
    cudaFree(c->plan);
    cudaFree(c->item_pages);
    cudaFree(c->d_free);
    cudaFree(c->d_small);
    cudaFree(c->part_o);
    cudaFree(c->part_ml);
}

// Wait for the cache's stream (the stream of its latest call; the caller
// keeps it alive).  Should the wait fail, wait for the device instead.
int wait_cache_stream(kv_cache* c)
{
    if (cudaStreamSynchronize(c->last_stream) != cudaSuccess) {
        cudaGetLastError();
        c->last_stream = nullptr;
        KVD_CUDA(cudaDeviceSynchronize());
    }
    return KVC_OK;
}

// Bring the host mirror up to the device after device-side steps or
// allocator calls.  Lazy: only calls that read the mirror (kv_seq_info,
// kv_cache_query, kv_cache_sync, host-planned steps, page order, enabling or
// disabling device steps) come here, and they wait for the cache's stream
// only, not the whole device; the state is then read back on the cache's own
// stream.
int sync_from_device(kv_cache* c)
{
    if (!c->dev_dirty) return KVC_OK;
    const kvc_config& k = c->cfg;
    std::vector<int32_t> pt((size_t)k.max_seqs * k.max_pages_per_seq), lens((size_t)k.max_seqs);
    int32_t small[2] = {0, 0};
    if (int rc = wait_cache_stream(c)) return rc;
    cudaStream_t st = c->copy_stream;
    KVD_CUDA(cudaMemcpyAsync(pt.data(), c->page_table(), pt.size() * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
    KVD_CUDA(cudaMemcpyAsync(lens.data(), c->seq_len_dev(), lens.size() * sizeof(int32_t), cudaMemcpyDeviceToHost,
                             st));
    KVD_CUDA(cudaMemcpyAsync(small, c->d_small, sizeof(small), cudaMemcpyDeviceToHost, st));
    KVD_CUDA(cudaStreamSynchronize(st));
    c->free_stack.assign((size_t)small[0], 0);
    if (small[0] > 0) {
        KVD_CUDA(cudaMemcpyAsync(c->free_stack.data(), c->d_free, (size_t)small[0] * sizeof(int32_t),
                                 cudaMemcpyDeviceToHost, st));
        KVD_CUDA(cudaStreamSynchronize(st));
    }
    c->pages_in_use = k.num_pages - small[0];
    for (int32_t s = 0; s < k.max_seqs; ++s) {
        if (c->lens[s] < 0) continue;
        c->lens[s] = lens[s];
        const int32_t np = (lens[s] + kPageSize - 1) / kPageSize;
        c->pages[s].assign(pt.begin() + (int64_t)s * k.max_pages_per_seq,
                           pt.begin() + (int64_t)s * k.max_pages_per_seq + np);
    }
    c->dev_dirty = false;
    return KVC_OK;
}

// After host-side allocator changes, the device free stack follows.
int push_free_stack(kv_cache* c, cudaStream_t st)
{
    if (!c->dev_mode) return KVC_OK;
    c->last_stream = st;
    const int32_t top = (int32_t)c->free_stack.size();
    if (top > 0)
        KVD_CUDA(cudaMemcpyAsync(c->d_free, c->free_stack.data(), (size_t)top * sizeof(int32_t),
                                 cudaMemcpyHostToDevice, st));
    KVD_CUDA(cudaMemcpyAsync(c->d_small, &top, sizeof(int32_t), cudaMemcpyHostToDevice, st));
    KVD_CUDA(cudaStreamSynchronize(st));   // the host buffers may change right after
    return KVC_OK;
}

}  // namespace

extern "C" {

const char* kv_last_error(void) { return g_last_error.c_str(); }

int kv_cache_create(const kvc_config* cfg, void* stream, kv_cache** out)
{
    if (!cfg || !out) return fail(KVC_ERR_INVALID, "kv_cache_create: null argument");
    *out = nullptr;
    const kvc_config& k = *cfg;
    if (k.num_layers < 1 || k.num_q_heads < 1 || k.num_kv_heads < 1 || k.head_dim < 1 ||
        k.page_size < 1 || k.max_seqs < 1 || k.max_pages_per_seq < 1 || k.num_pages < 1)
        return fail(KVC_ERR_INVALID, "kv_cache_create: every size must be positive");
    if (k.num_q_heads % k.num_kv_heads != 0)
        return fail(KVC_ERR_INVALID, "kv_cache_create: num_q_heads must be a multiple of num_kv_heads");
    if (k.num_q_heads / k.num_kv_heads > kMaxGroup)
        return fail(KVC_ERR_UNSUPPORTED, "kv_cache_create: more than 8 query heads per KV head");
    if (k.head_dim != 64 && k.head_dim != 128)
        return fail(KVC_ERR_UNSUPPORTED, "kv_cache_create: head_dim must be 64 or 128");
    if (k.page_size != kPageSize) return fail(KVC_ERR_UNSUPPORTED, "kv_cache_create: page_size must be 16");
    if (k.max_seqs > 65535) return fail(KVC_ERR_INVALID, "kv_cache_create: max_seqs > 65535");
    if ((int64_t)k.max_seqs * k.max_pages_per_seq + k.max_seqs >= (int64_t)1 << 31)
        return fail(KVC_ERR_INVALID, "kv_cache_create: page table larger than 2^31 entries");
    if (k.num_pages * k.num_kv_heads * kPageSize >= (int64_t)1 << 31)
        return fail(KVC_ERR_INVALID, "kv_cache_create: num_pages * num_kv_heads * 16 must be < 2^31");
    if (k.flags & ~KVC_FLAG_HOST_ONLY) return fail(KVC_ERR_INVALID, "kv_cache_create: unknown flag");

    kv_cache* c = new kv_cache();
    c->cfg = k;
    c->host_only = (k.flags & KVC_FLAG_HOST_ONLY) != 0;
    c->group = k.num_q_heads / k.num_kv_heads;
    c->lens.assign(k.max_seqs, -1);
    c->pages.assign(k.max_seqs, {});
    c->stamp.assign(k.max_seqs, 0);
    c->free_stack.resize(k.num_pages);
    for (int64_t i = 0; i < k.num_pages; ++i) c->free_stack[i] = (int32_t)(k.num_pages - 1 - i);

    if (!c->host_only) {
        cudaStream_t st = static_cast<cudaStream_t>(stream);
        auto bail = [&](int rc) {
            release_device(c);
            delete c;
            return rc;
        };
#define KVD_CUDA_C(call)                                                                    \
    do {                                                                                    \
        cudaError_t e_ = (call);                                                            \
        if (e_ != cudaSuccess)                                                              \
            return bail(fail(e_ == cudaErrorMemoryAllocation ? KVC_ERR_OOM : KVC_ERR_CUDA,  \
                             std::string(#call) + ": " + cudaGetErrorString(e_)));         \
    } while (0)
        KVD_CUDA_C(cudaGetDevice(&c->device));
        KVD_CUDA_C(cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking));
        c->last_stream = st;
        KVD_CUDA_C(cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device));
        KVD_CUDA_C(decode_variant_info(k.head_dim, c->group > 1, &c->variant));
        auto encode = tensor_map_encoder();
        if (!encode) return bail(fail(KVC_ERR_CUDA, "kv_cache_create: cuTensorMapEncodeTiled unavailable"));

        c->layer_elems = (size_t)k.num_pages * k.num_kv_heads * kPageSize * k.head_dim;
        const size_t pool_bytes = 2 * (size_t)k.num_layers * c->layer_elems * sizeof(uint16_t);
        const size_t meta_elems = (size_t)k.max_seqs * k.max_pages_per_seq + k.max_seqs;
        KVD_CUDA_C(cudaMalloc((void**)&c->pools, pool_bytes));
        KVD_CUDA_C(cudaMalloc((void**)&c->meta, meta_elems * sizeof(int32_t)));
        KVD_CUDA_C(cudaMalloc((void**)&c->step_seq, (size_t)k.max_seqs * sizeof(int32_t)));
        KVD_CUDA_C(cudaMalloc((void**)&c->rows, (size_t)k.max_seqs * sizeof(int2)));
        KVD_CUDA_C(cudaMalloc((void**)&c->queue, 4 * sizeof(uint32_t)));
        KVD_CUDA_C(cudaMalloc((void**)&c->start_flags, (size_t)c->num_sms * 32 * sizeof(uint32_t)));
        KVD_CUDA_C(cudaMalloc((void**)&c->step_no, sizeof(uint32_t)));
        KVD_CUDA_C(cudaMemsetAsync(c->start_flags, 0, (size_t)c->num_sms * 32 * sizeof(uint32_t), st));
        KVD_CUDA_C(cudaMemsetAsync(c->step_no, 0, sizeof(uint32_t), st));
        KVD_CUDA_C(cudaMalloc((void**)&c->err, sizeof(int32_t)));
        KVD_CUDA_C(cudaMemsetAsync(c->pools, 0, pool_bytes, st));
        KVD_CUDA_C(cudaMemsetAsync(c->meta, 0xff, (size_t)k.max_seqs * k.max_pages_per_seq * sizeof(int32_t), st));
        KVD_CUDA_C(cudaMemsetAsync(c->seq_len_dev(), 0, (size_t)k.max_seqs * sizeof(int32_t), st));
        KVD_CUDA_C(cudaMemsetAsync(c->step_seq, 0, (size_t)k.max_seqs * sizeof(int32_t), st));
        KVD_CUDA_C(cudaMemsetAsync(c->rows, 0, (size_t)k.max_seqs * sizeof(int2), st));
        KVD_CUDA_C(cudaMemsetAsync(c->queue, 0, 4 * sizeof(uint32_t), st));
        KVD_CUDA_C(cudaMemsetAsync(c->err, 0, sizeof(int32_t), st));
#undef KVD_CUDA_C

        // One TMA view per layer covering its K and V pools: a page's
        // (page, head) tiles of K and V arrive with a single load.
        c->tmaps.resize((size_t)k.num_layers);
        for (int l = 0; l < k.num_layers; ++l) {
            const int64_t v_stride = (int64_t)((char*)c->v_pool(l) - (char*)c->k_pool(l));
            CUresult r = encode_tile_map(reinterpret_cast<void*>(encode), &c->tmaps[l], c->k_pool(l),
                                         k.num_pages * k.num_kv_heads * kPageSize, k.head_dim, v_stride);
            if (r != CUDA_SUCCESS) {
                release_device(c);
                delete c;
                return fail(KVC_ERR_CUDA, "kv_cache_create: cuTensorMapEncodeTiled failed (" + std::to_string((int)r) +
                                              ")");
            }
        }
    }
    *out = c;
    return KVC_OK;
}

int kv_cache_destroy(kv_cache* c)
{
    if (!c) return KVC_OK;
    int rc = KVC_OK;
    if (!c->host_only) {
        cudaError_t e = cudaDeviceSynchronize();
        if (e != cudaSuccess) rc = fail(KVC_ERR_CUDA, std::string("kv_cache_destroy: ") + cudaGetErrorString(e));
        release_device(c);
    }
    delete c;
    return rc;
}

int kv_cache_set_page_order(kv_cache* c, const int32_t* order, int64_t n)
{
    if (!c || !order) return fail(KVC_ERR_INVALID, "kv_cache_set_page_order: null argument");
    if (int rc = sync_from_device(c)) return rc;
    if (n != c->cfg.num_pages) return fail(KVC_ERR_INVALID, "kv_cache_set_page_order: n must equal num_pages");
    if (c->pages_in_use) return fail(KVC_ERR_INVALID, "kv_cache_set_page_order: pages are in use");
    std::vector<uint8_t> seen((size_t)n, 0);
    for (int64_t i = 0; i < n; ++i) {
        if (order[i] < 0 || order[i] >= n || seen[order[i]])
            return fail(KVC_ERR_INVALID, "kv_cache_set_page_order: not a permutation of the pool");
        seen[order[i]] = 1;
    }
    for (int64_t i = 0; i < n; ++i) c->free_stack[i] = order[n - 1 - i];
    return push_free_stack(c, nullptr);
}

int kv_cache_query(kv_cache* c, kvc_stats* s)
{
    if (!c || !s) return fail(KVC_ERR_INVALID, "kv_cache_query: null argument");
    if (int rc = sync_from_device(c)) return rc;
    const kvc_config& k = c->cfg;
    s->pages_in_use = c->pages_in_use;
    s->free_pages = (int64_t)c->free_stack.size();
    s->kv_bytes_allocated = 2 * (int64_t)k.num_layers * k.num_kv_heads * k.head_dim * 2 * kPageSize * c->pages_in_use;
    s->pool_bytes = c->host_only ? 0 : (int64_t)(2 * (size_t)k.num_layers * c->layer_elems * sizeof(uint16_t));
    s->live_seqs = c->live;
    s->device_error = 0;
    s->kernel_launches = c->launches;
    if (c->host_only) return KVC_OK;
    if (int rc = wait_cache_stream(c)) return rc;
    KVD_CUDA(cudaMemcpyAsync(&s->device_error, c->err, sizeof(int32_t), cudaMemcpyDeviceToHost, c->copy_stream));
    KVD_CUDA(cudaStreamSynchronize(c->copy_stream));
    if (s->device_error & (KVC_DEVERR_PAGE_RANGE | KVC_DEVERR_SEQ_RANGE))
        return fail(KVC_ERR_PAGE_TABLE, "device found a page id or length outside its range");
    if (s->device_error & KVC_DEVERR_OOM) return fail(KVC_ERR_OOM, "a device-side step found the page pool exhausted");
    if (s->device_error) return fail(KVC_ERR_DEVICE, "a device-side pipeline wait gave up");
    return KVC_OK;
}

int kv_cache_pool(kv_cache* c, int32_t layer, void** k_pool, void** v_pool)
{
    if (!c || !k_pool || !v_pool) return fail(KVC_ERR_INVALID, "kv_cache_pool: null argument");
    if (int rc = check_device(c, "kv_cache_pool")) return rc;
    if (layer < 0 || layer >= c->cfg.num_layers) return fail(KVC_ERR_INVALID, "kv_cache_pool: bad layer");
    *k_pool = c->k_pool(layer);
    *v_pool = c->v_pool(layer);
    return KVC_OK;
}

int kv_cache_set_split_pages(kv_cache* c, int32_t pages)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_cache_set_split_pages: null cache");
    if (pages < 0 || pages > kMaxItemPages)
        return fail(KVC_ERR_INVALID, "kv_cache_set_split_pages: pages must be in 0 .. 1024");
    c->split_override = pages;
    return KVC_OK;
}

int kv_seq_create(kv_cache* c, int32_t* seq_id)
{
    if (!c || !seq_id) return fail(KVC_ERR_INVALID, "kv_seq_create: null argument");
    for (int32_t i = 0; i < c->cfg.max_seqs; ++i) {
        if (c->lens[i] < 0) {
            c->lens[i] = 0;
            c->pages[i].clear();
            ++c->live;
            *seq_id = i;
            return KVC_OK;
        }
    }
    return fail(KVC_ERR_OOM, "kv_seq_create: every sequence slot is in use");
}

// With device-side steps the device holds the free stack, lengths and page
// table: a reservation or release is a stream-ordered kernel, with no host
// synchronisation; its failures (full page row, exhausted pool) set device
// error bits instead of a return code.
static int seq_op_device(kv_cache* c, int32_t seq, int32_t n, bool free_seq, void* stream)
{
    SeqOpArgs a;
    a.free_seq = free_seq ? 1 : 0;
    a.seq = seq;
    a.n = n;
    a.max_pages = c->cfg.max_pages_per_seq;
    a.free_pages = c->d_free;
    a.free_top = c->d_small;
    a.seq_len = c->seq_len_dev();
    a.page_table = c->page_table();
    a.err = c->err;
    c->last_stream = static_cast<cudaStream_t>(stream);
    KVD_CUDA(launch_seq_op(a, c->last_stream));
    ++c->launches;
    c->dev_dirty = true;
    return KVC_OK;
}

int kv_seq_reserve(kv_cache* c, int32_t seq, int32_t n, void* stream)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_seq_reserve: null cache");
    if (c->dev_mode) {
        if (int rc = check_seq(c, seq)) return rc;
        if (n < 0 || (int64_t)n > (int64_t)c->cfg.max_pages_per_seq * kPageSize)
            return fail(KVC_ERR_INVALID, "kv_seq_reserve: token count outside 0 .. max_pages_per_seq * 16");
        if (n == 0) return KVC_OK;
        return seq_op_device(c, seq, n, false, stream);
    }
    if (int rc = sync_from_device(c)) return rc;
    if (int rc = check_seq(c, seq)) return rc;
    if (n < 0) return fail(KVC_ERR_INVALID, "kv_seq_reserve: negative token count");
    const int64_t len = c->lens[seq], new_len = len + n;
    const int64_t have = (len + kPageSize - 1) / kPageSize, need = (new_len + kPageSize - 1) / kPageSize;
    if (need > c->cfg.max_pages_per_seq) return fail(KVC_ERR_INVALID, "kv_seq_reserve: page-table row too short");
    if (need - have > (int64_t)c->free_stack.size()) return fail(KVC_ERR_OOM, "kv_seq_reserve: page pool exhausted");
    if (n == 0) return KVC_OK;
    std::vector<int32_t> idx, val;
    for (int64_t p = have; p < need; ++p) {
        const int32_t page = c->pop_page();
        c->pages[seq].push_back(page);
        idx.push_back(seq * c->cfg.max_pages_per_seq + (int32_t)p);
        val.push_back(page);
    }
    c->lens[seq] = (int32_t)new_len;
    idx.push_back(c->seq_len_index(seq));
    val.push_back((int32_t)new_len);
    if (int rc = push_updates(c, idx, val, static_cast<cudaStream_t>(stream))) return rc;
    return push_free_stack(c, static_cast<cudaStream_t>(stream));
}

int kv_seq_free(kv_cache* c, int32_t seq, void* stream)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_seq_free: null cache");
    if (c->dev_mode) {
        if (int rc = check_seq(c, seq)) return rc;
        if (int rc = seq_op_device(c, seq, 0, true, stream)) return rc;
        c->lens[seq] = -1;   // the id is free again; its pages and length are the device's
        c->pages[seq].clear();
        --c->live;
        c->step_active = false;
        return KVC_OK;
    }
    if (int rc = sync_from_device(c)) return rc;
    if (int rc = check_seq(c, seq)) return rc;
    std::vector<int32_t> idx, val;
    auto& pg = c->pages[seq];
    for (size_t i = 0; i < pg.size(); ++i) {
        idx.push_back(seq * c->cfg.max_pages_per_seq + (int32_t)i);
        val.push_back(-1);
    }
    for (size_t i = pg.size(); i-- > 0;) c->free_stack.push_back(pg[i]);
    c->pages_in_use -= (int64_t)pg.size();
    pg.clear();
    c->lens[seq] = -1;
    --c->live;
    c->step_active = false;
    idx.push_back(c->seq_len_index(seq));
    val.push_back(0);
    if (int rc = push_updates(c, idx, val, static_cast<cudaStream_t>(stream))) return rc;
    return push_free_stack(c, static_cast<cudaStream_t>(stream));
}

int kv_seq_info(kv_cache* c, int32_t seq, int32_t* len, int32_t* page_ids, int32_t capacity, int32_t* n_pages)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_seq_info: null cache");
    if (int rc = sync_from_device(c)) return rc;
    if (int rc = check_seq(c, seq)) return rc;
    const auto& pg = c->pages[seq];
    if (len) *len = c->lens[seq];
    if (n_pages) *n_pages = (int32_t)pg.size();
    if (page_ids)
        for (int32_t i = 0; i < capacity && i < (int32_t)pg.size(); ++i) page_ids[i] = pg[i];
    return KVC_OK;
}

static int token_copy(kv_cache* c, const char* what, int32_t layer, int32_t seq, int32_t first, int32_t n,
                      void* k, void* v, int to_pool, void* stream)
{
    if (!c) return fail(KVC_ERR_INVALID, std::string(what) + ": null cache");
    if (int rc = check_device(c, what)) return rc;
    if (int rc = check_seq(c, seq)) return rc;
    if (layer < 0 || layer >= c->cfg.num_layers) return fail(KVC_ERR_INVALID, std::string(what) + ": bad layer");
    // With device-side steps the length lives on the device: the kernel
    // checks the positions (bit 4 if they pass it); otherwise the host does.
    const int64_t limit = c->dev_mode ? (int64_t)c->cfg.max_pages_per_seq * kPageSize : c->lens[seq];
    if (first < 0 || n < 0 || (int64_t)first + n > limit)
        return fail(KVC_ERR_INVALID, std::string(what) + ": positions outside the reserved length");
    if (n == 0) return KVC_OK;
    if (!k || !v || !aligned16(k) || !aligned16(v))
        return fail(KVC_ERR_INVALID, std::string(what) + ": k / v must be non-null and 16-byte aligned");
    TokenCopyArgs a;
    a.pool_k = c->k_pool(layer);
    a.pool_v = c->v_pool(layer);
    a.pt_row = c->page_table() + (int64_t)seq * c->cfg.max_pages_per_seq;
    a.len = c->dev_mode ? c->seq_len_dev() + seq : nullptr;
    a.num_pages = c->cfg.num_pages;
    a.H_kv = c->cfg.num_kv_heads;
    a.D = c->cfg.head_dim;
    a.first_pos = first;
    a.n = n;
    a.tok_k = static_cast<uint16_t*>(k);
    a.tok_v = static_cast<uint16_t*>(v);
    a.to_pool = to_pool;
    a.err = c->err;
    c->last_stream = static_cast<cudaStream_t>(stream);
    KVD_CUDA(launch_token_copy(a, static_cast<cudaStream_t>(stream)));
    ++c->launches;
    return KVC_OK;
}

int kv_write_tokens(kv_cache* c, int32_t layer, int32_t seq, int32_t first_pos, int32_t n, const void* k,
                    const void* v, void* stream)
{
    return token_copy(c, "kv_write_tokens", layer, seq, first_pos, n, const_cast<void*>(k), const_cast<void*>(v), 1,
                      stream);
}

int kv_read_tokens(kv_cache* c, int32_t layer, int32_t seq, int32_t first_pos, int32_t n, void* k_out, void* v_out,
                   void* stream)
{
    return token_copy(c, "kv_read_tokens", layer, seq, first_pos, n, k_out, v_out, 0, stream);
}

int kv_write_varlen(kv_cache* c, int32_t layer_first, int32_t n_layers, int32_t n_blocks, const int32_t* seq_ids,
                    const int32_t* first_pos, const int32_t* cu_seqlens, const void* k, const void* v, void* stream)
{
    if (!c || (n_blocks > 0 && (!seq_ids || !cu_seqlens)))
        return fail(KVC_ERR_INVALID, "kv_write_varlen: null argument");
    if (n_layers < 1 || n_layers > 65535 || layer_first < 0 || (int64_t)layer_first + n_layers > c->cfg.num_layers)
        return fail(KVC_ERR_INVALID, "kv_write_varlen: layers outside the cache");
    if (n_blocks < 0) return fail(KVC_ERR_INVALID, "kv_write_varlen: negative block count");
    if (n_blocks == 0) return KVC_OK;
    if (cu_seqlens[0] != 0) return fail(KVC_ERR_INVALID, "kv_write_varlen: cu_seqlens[0] must be 0");
    std::vector<int32_t> order((size_t)n_blocks);
    for (int32_t i = 0; i < n_blocks; ++i) {
        if (int rc = check_seq(c, seq_ids[i])) return rc;
        const int64_t n = (int64_t)cu_seqlens[i + 1] - cu_seqlens[i];
        const int64_t f = first_pos ? first_pos[i] : 0;
        if (n < 0) return fail(KVC_ERR_INVALID, "kv_write_varlen: cu_seqlens must not decrease");
        // with device-side steps the kernel checks against the device's length
        const int64_t limit = c->dev_mode ? (int64_t)c->cfg.max_pages_per_seq * kPageSize : c->lens[seq_ids[i]];
        if (f < 0 || f + n > limit)
            return fail(KVC_ERR_INVALID, "kv_write_varlen: positions outside the reserved length");
        order[i] = i;
    }
    // Two blocks may not write the same position of a sequence.
    auto fpos = [&](int32_t i) { return first_pos ? first_pos[i] : 0; };
    std::sort(order.begin(), order.end(), [&](int32_t x, int32_t y) {
        return seq_ids[x] != seq_ids[y] ? seq_ids[x] < seq_ids[y] : fpos(x) < fpos(y);
    });
    int64_t end = 0;   // end of the blocks seen so far in the current sequence
    for (int32_t j = 0; j < n_blocks; ++j) {
        const int32_t y = order[j];
        const int64_t n = (int64_t)cu_seqlens[y + 1] - cu_seqlens[y];
        if (j == 0 || seq_ids[order[j - 1]] != seq_ids[y]) end = 0;
        if (n == 0) continue;
        if (fpos(y) < end) return fail(KVC_ERR_INVALID, "kv_write_varlen: blocks overlap in a sequence");
        end = fpos(y) + n;
    }
    const int64_t rows = cu_seqlens[n_blocks];
    if (rows == 0) return KVC_OK;
    if (!k || !v || !aligned16(k) || !aligned16(v))
        return fail(KVC_ERR_INVALID, "kv_write_varlen: k / v must be non-null and 16-byte aligned");
    if (int rc = check_device(c, "kv_write_varlen")) return rc;

    VarlenWriteArgs a;
    a.pool_k = c->k_pool(layer_first);
    a.pool_v = c->v_pool(layer_first);
    a.pool_layer_stride = (int64_t)c->layer_elems;
    a.k = static_cast<const uint16_t*>(k);
    a.v = static_cast<const uint16_t*>(v);
    a.src_layer_stride = rows * c->cfg.num_kv_heads * c->cfg.head_dim;
    a.page_table = c->page_table();
    a.seq_len = c->dev_mode ? c->seq_len_dev() : nullptr;
    a.num_pages = c->cfg.num_pages;
    a.max_pages = c->cfg.max_pages_per_seq;
    a.H_kv = c->cfg.num_kv_heads;
    a.D = c->cfg.head_dim;
    a.err = c->err;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    c->last_stream = st;
    // Blocks go kVarlenMax at a time (empty ones skipped), one launch each.
    auto flush = [&]() -> int {
        if (a.n_blocks == 0) return KVC_OK;
        a.n_tiles = a.tile_start[a.n_blocks];
        KVD_CUDA(launch_varlen_write(a, n_layers, st));
        ++c->launches;
        a.n_blocks = 0;
        return KVC_OK;
    };
    a.n_blocks = 0;
    a.tile_start[0] = 0;
    for (int32_t i = 0; i < n_blocks; ++i) {
        const int32_t n = cu_seqlens[i + 1] - cu_seqlens[i];
        if (n == 0) continue;
        const int32_t f = fpos(i);
        const int32_t j = a.n_blocks;
        a.seq[j] = seq_ids[i];
        a.first_pos[j] = f;
        a.n_tok[j] = n;
        a.src_row[j] = cu_seqlens[i];
        a.tile_start[j + 1] = a.tile_start[j] + ((f + n - 1) / kPageSize - f / kPageSize + 1);
        if (++a.n_blocks == kVarlenMax)
            if (int rc = flush()) return rc;
    }
    return flush();
}

int kv_begin_step(kv_cache* c, int32_t batch, const int32_t* seq_ids, void* stream)
{
    if (!c || !seq_ids) return fail(KVC_ERR_INVALID, "kv_begin_step: null argument");
    if (int rc = sync_from_device(c)) return rc;
    if (batch < 1 || batch > c->cfg.max_seqs) return fail(KVC_ERR_INVALID, "kv_begin_step: batch outside 1 .. max_seqs");
    if (++c->stamp_gen == 0) {
        std::fill(c->stamp.begin(), c->stamp.end(), 0u);
        c->stamp_gen = 1;
    }
    int64_t need = 0;
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t s = seq_ids[b];
        if (int rc = check_seq(c, s)) return rc;
        if (c->stamp[s] == c->stamp_gen) return fail(KVC_ERR_INVALID, "kv_begin_step: sequence listed twice");
        c->stamp[s] = c->stamp_gen;
        const int64_t len = c->lens[s];
        if ((len + 1 + kPageSize - 1) / kPageSize > c->cfg.max_pages_per_seq)
            return fail(KVC_ERR_INVALID, "kv_begin_step: page-table row too short");
        if (len % kPageSize == 0) ++need;
    }
    if (need > (int64_t)c->free_stack.size()) return fail(KVC_ERR_OOM, "kv_begin_step: page pool exhausted");

    // Size the plan from the lengths after this step, before changing anything.
    std::vector<int32_t> np_after((size_t)batch);
    int64_t total_units = 0;
    for (int32_t b = 0; b < batch; ++b) {
        np_after[b] = (c->lens[seq_ids[b]] + 1 + kPageSize - 1) / kPageSize;
        total_units += (int64_t)np_after[b] * c->cfg.num_kv_heads;
    }
    const int32_t T = c->split_override ? c->split_override : auto_item_pages(c, total_units);
    // Plan order: longest rows first (stable), when the batch fits one launch.
    const bool use_order = batch <= kPatchMax;
    std::vector<int32_t> order((size_t)batch), rank((size_t)batch);
    for (int32_t b = 0; b < batch; ++b) order[b] = b;
    if (use_order)
        std::stable_sort(order.begin(), order.end(),
                         [&](int32_t x, int32_t y) { return np_after[x] > np_after[y]; });
    for (int32_t i = 0; i < batch; ++i) rank[order[i]] = i;
    const int32_t cap = chunk_cap(c, batch, *std::max_element(np_after.begin(), np_after.end()), T);
    int64_t entries = 0;
    int32_t stride = 1;
    bool split = false;
    int32_t max_chunks = 1;
    for (int32_t b = 0; b < batch; ++b) {
        const int nch = row_chunks(np_after[b], row_item_pages(T, rank[b], batch), cap);
        entries += nch;
        split = split || nch > 1;
        max_chunks = std::max(max_chunks, nch);
        stride = std::max(stride, (np_after[b] + nch - 1) / nch);
    }
    if (!c->host_only)
        if (int rc = grow_scratch(c, entries, entries * c->cfg.num_kv_heads, entries * stride,
                                  static_cast<cudaStream_t>(stream)))
            return rc;

    // Host mirror: every sequence of the batch gets position len.
    std::vector<int32_t> new_page((size_t)batch, -1);
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t s = seq_ids[b];
        if (c->lens[s] % kPageSize == 0) {
            new_page[b] = c->pop_page();
            c->pages[s].push_back(new_page[b]);
        }
        c->lens[s] += 1;
    }
    c->step_active = false;
    if (!c->host_only) {
        cudaStream_t st = static_cast<cudaStream_t>(stream);
        c->last_stream = st;
        StepPatch patch;
        PlanArgs pa;
        pa.batch = batch;
        pa.item_pages = T;
        pa.max_pages = c->cfg.max_pages_per_seq;
        pa.step_seq = c->step_seq;
        pa.seq_len = c->seq_len_dev();
        pa.page_table = c->page_table();
        pa.plan = c->plan;
        pa.rows = c->rows;
        pa.chunk_cap = cap;
        pa.page_ids = c->item_pages;
        pa.page_stride = stride;
        pa.err = c->err;
        pa.step_no = c->step_no;
        // Longest rows first: their items start early and the tail is short.
        pa.use_order = use_order ? 1 : 0;
        if (use_order)
            for (int32_t i = 0; i < batch; ++i) pa.order[i] = order[i];
        for (int32_t b0 = 0; b0 < batch; b0 += kPatchMax) {
            const int32_t n = std::min(kPatchMax, batch - b0);
            patch.n = n;
            patch.b0 = b0;
            for (int32_t i = 0; i < n; ++i) {
                patch.seq[i] = seq_ids[b0 + i];
                patch.new_len[i] = c->lens[seq_ids[b0 + i]];
                patch.new_page[i] = new_page[b0 + i];
            }
            pa.build = (b0 + n == batch) ? 1 : 0;
            KVD_CUDA(launch_step(patch, pa, st));
            ++c->launches;
        }
    }
    if (!c->host_only)
        if (int rc = push_free_stack(c, static_cast<cudaStream_t>(stream))) return rc;
    c->attn_tag = 0;
    c->prev_merge = false;
    c->step_active = true;
    c->step_dev = false;
    c->step_split = split;
    c->step_max_chunks = max_chunks;
    c->page_stride = stride;
    c->step_batch = batch;
    c->step_entries = (int32_t)entries;
    return KVC_OK;
}

static int check_step(kv_cache* c, const char* what, int32_t layer, int32_t batch)
{
    if (!c) return fail(KVC_ERR_INVALID, std::string(what) + ": null cache");
    if (int rc = check_device(c, what)) return rc;
    if (!c->step_active) return fail(KVC_ERR_INVALID, std::string(what) + ": no decode step is active");
    if (batch != c->step_batch) return fail(KVC_ERR_INVALID, std::string(what) + ": batch differs from the step's");
    if (layer < 0 || layer >= c->cfg.num_layers) return fail(KVC_ERR_INVALID, std::string(what) + ": bad layer");
    return KVC_OK;
}

int kv_append(kv_cache* c, int32_t layer, int32_t batch, const void* k_new, const void* v_new, void* stream)
{
    if (int rc = check_step(c, "kv_append", layer, batch)) return rc;
    if (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))
        return fail(KVC_ERR_INVALID, "kv_append: k_new / v_new must be non-null and 16-byte aligned");
    AppendArgs a;
    a.pool_k = c->k_pool(layer);
    a.pool_v = c->v_pool(layer);
    a.k_new = static_cast<const uint16_t*>(k_new);
    a.v_new = static_cast<const uint16_t*>(v_new);
    a.step_seq = c->step_seq;
    a.seq_len = c->seq_len_dev();
    a.page_table = c->page_table();
    a.num_pages = c->cfg.num_pages;
    a.batch = batch;
    a.H_kv = c->cfg.num_kv_heads;
    a.D = c->cfg.head_dim;
    a.max_pages = c->cfg.max_pages_per_seq;
    a.err = c->err;
    c->last_stream = static_cast<cudaStream_t>(stream);
    KVD_CUDA(launch_append(a, static_cast<cudaStream_t>(stream)));
    ++c->launches;
    return KVC_OK;
}

static int launch_attention(kv_cache* c, const char* what, int32_t layer, int32_t batch, const void* q,
                            const void* k_new, const void* v_new, void* out, float softmax_scale, void* stream)
{
    if (int rc = check_step(c, what, layer, batch)) return rc;
    const bool fused = k_new != nullptr;
    if (!q || !out || !aligned16(q) || !aligned16(out))
        return fail(KVC_ERR_INVALID, std::string(what) + ": q / out must be non-null and 16-byte aligned");
    if (fused && (!v_new || !aligned16(k_new) || !aligned16(v_new)))
        return fail(KVC_ERR_INVALID, std::string(what) + ": k_new / v_new must be non-null and 16-byte aligned");
    if (!(softmax_scale <= 0.f) && !std::isfinite(softmax_scale))
        return fail(KVC_ERR_INVALID, std::string(what) + ": softmax_scale must be finite");
    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt((float)c->cfg.head_dim);
    DecodeParams p;
    p.q = static_cast<const uint16_t*>(q);
    p.out = static_cast<uint16_t*>(out);
    p.page_table = c->page_table();
    p.plan = c->plan;
    p.part_o = c->part_o;
    p.part_ml = c->part_ml;
    p.rows = c->rows;
    p.item_pages = c->item_pages;
    p.page_stride = c->page_stride;
    p.n_entries_dev = c->step_dev ? c->d_small + 1 : nullptr;
    p.batch = batch;
    // Consecutive attention launches use different work counters: a chained
    // launch may start while the previous one drains, and each launch resets
    // the counter of the next one once the previous launch has completed.
    p.queue = c->queue + (c->attn_launches & 1u);
    p.queue_next = c->queue + ((c->attn_launches + 1u) & 1u);
    p.err = c->err;
    p.num_pages = c->cfg.num_pages;
    p.n_items = c->step_entries * c->cfg.num_kv_heads;
    p.H_kv = c->cfg.num_kv_heads;
    p.H_q = c->cfg.num_q_heads;
    p.G = c->group;
    p.max_pages = c->cfg.max_pages_per_seq;
    p.scale_log2 = scale * 1.4426950408889634f;
    p.k_new = static_cast<const uint16_t*>(k_new);
    p.v_new = static_cast<const uint16_t*>(v_new);
    p.pool_k = c->k_pool(layer);
    p.pool_v = c->v_pool(layer);
    const int64_t resident = (int64_t)c->num_sms * std::max(1, c->variant.ctas_per_sm);
    const int64_t want = (p.n_items + c->variant.warps - 1) / c->variant.warps;
    const int grid = (int)std::max<int64_t>(1, std::min(resident, want));
    p.kv_map = 1;
    const bool pdl = fused && c->chain_launches == c->launches && c->chain_stream == stream;
    // The early L2 start waits for the previous launch's merge pass, so only
    // a launch chained after one that has a merge pass looks for it, and only
    // when both were issued the same way: eagerly, or into the same stream
    // capture (a graph replays its own launches in order, but what precedes
    // a graph's first launch at replay is not what preceded it at capture).
    unsigned long long capture = 0;
    {
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if (cudaStreamGetCaptureInfo(static_cast<cudaStream_t>(stream), &cs, &capture) != cudaSuccess ||
            cs != cudaStreamCaptureStatusActive)
            capture = 0;
        cudaGetLastError();
    }
    p.start_flags = c->start_flags;
    p.step_no = c->step_no;
    p.prev_tag = (pdl && c->prev_merge && capture == c->prev_capture) ? c->attn_tag : 0;
    c->prev_capture = capture;
    p.tag = ++c->attn_tag;
    p.num_sms = c->num_sms;
    c->last_stream = static_cast<cudaStream_t>(stream);
    KVD_CUDA(launch_decode(c->cfg.head_dim, c->group > 1, fused, pdl, grid, c->tmaps[layer], c->tmaps[layer], p,
                           static_cast<cudaStream_t>(stream)));
    ++c->launches;
    ++c->attn_launches;   // the launch used one counter and resets the other, whatever follows
    c->prev_merge = false;
    if (c->step_split) {
        // Launched early (fused), the merge CTAs sit beside the resident split pass.
        const int split_regs =
            fused ? ((c->variant.ctas_per_sm * c->variant.warps + 3) / 4) * warp_register_allocation(c->variant.regs)
                  : 0;
        KVD_CUDA(launch_merge(c->cfg.head_dim, fused, c->step_max_chunks, c->num_sms, split_regs, p,
                              static_cast<cudaStream_t>(stream)));
        ++c->launches;
        c->prev_merge = true;
    }
    c->chain_launches = c->launches;
    c->chain_stream = stream;
    return KVC_OK;
}

int decode_attention(kv_cache* c, int32_t layer, int32_t batch, const void* q, void* out, float softmax_scale,
                     void* stream)
{
    return launch_attention(c, "decode_attention", layer, batch, q, nullptr, nullptr, out, softmax_scale, stream);
}

int decode_attention_append(kv_cache* c, int32_t layer, int32_t batch, const void* q, const void* k_new,
                            const void* v_new, void* out, float softmax_scale, void* stream)
{
    if (!k_new) return fail(KVC_ERR_INVALID, "decode_attention_append: k_new must be non-null");
    return launch_attention(c, "decode_attention_append", layer, batch, q, k_new, v_new, out, softmax_scale, stream);
}

int kv_cache_device_steps(kv_cache* c, int32_t max_batch, int32_t enable, void* stream)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_cache_device_steps: null cache");
    if (int rc = check_device(c, "kv_cache_device_steps")) return rc;
    if (int rc = sync_from_device(c)) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    c->step_active = false;
    if (!enable) {
        c->dev_mode = false;
        return KVC_OK;
    }
    if (max_batch < 1 || max_batch > c->cfg.max_seqs)
        return fail(KVC_ERR_INVALID, "kv_cache_device_steps: max_batch outside 1 .. max_seqs");
    c->dev_mode = false;   // (re-)enabling may resize the buffers
    // Work-item size from the pages now held (steps add a token per sequence).
    const int32_t T = c->split_override
                          ? c->split_override
                          : auto_item_pages(c, c->pages_in_use * (int64_t)c->cfg.num_kv_heads);
    const int32_t cap = chunk_cap(c, max_batch, c->cfg.max_pages_per_seq, T);
    const int32_t entries = max_batch * cap;
    const int32_t stride = std::max(T, (c->cfg.max_pages_per_seq + cap - 1) / cap) + 1;
    if (int rc = grow_scratch(c, entries, (int64_t)entries * c->cfg.num_kv_heads, (int64_t)entries * stride, st))
        return rc;
    if (!c->d_free) KVD_CUDA(cudaMalloc((void**)&c->d_free, (size_t)c->cfg.num_pages * sizeof(int32_t)));
    if (!c->d_small) KVD_CUDA(cudaMalloc((void**)&c->d_small, 2 * sizeof(int32_t)));
    c->dev_mode = true;
    c->dev_max_batch = max_batch;
    c->dev_item_pages = T;
    c->dev_entries_cap = entries;
    c->dev_stride = stride;
    c->dev_chunk_cap = cap;
    return push_free_stack(c, st);
}

int kv_begin_step_device(kv_cache* c, int32_t batch, const int32_t* seq_ids, void* stream)
{
    if (!c || !seq_ids) return fail(KVC_ERR_INVALID, "kv_begin_step_device: null argument");
    if (!c->dev_mode) return fail(KVC_ERR_INVALID, "kv_begin_step_device: device steps are not enabled");
    if (batch < 1 || batch > c->dev_max_batch)
        return fail(KVC_ERR_INVALID, "kv_begin_step_device: batch outside 1 .. max_batch");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    StepDevArgs a;
    a.batch = batch;
    a.max_seqs = c->cfg.max_seqs;
    a.item_pages = c->dev_item_pages;
    a.max_pages = c->cfg.max_pages_per_seq;
    a.max_entries = c->dev_entries_cap;
    a.seq_ids = seq_ids;
    a.free_pages = c->d_free;
    a.free_top = c->d_small;
    a.step_seq = c->step_seq;
    a.seq_len = c->seq_len_dev();
    a.page_table = c->page_table();
    a.plan = c->plan;
    a.rows = c->rows;
    a.n_entries = c->d_small + 1;
    a.chunk_cap = c->dev_chunk_cap;
    a.page_ids = c->item_pages;
    a.page_stride = c->dev_stride;
    a.err = c->err;
    a.step_no = c->step_no;
    c->last_stream = st;
    KVD_CUDA(launch_step_device(a, st));
    ++c->launches;
    c->dev_dirty = true;
    c->attn_tag = 0;
    c->prev_merge = false;
    c->step_active = true;
    c->step_dev = true;
    c->step_split = true;   // the row split is only known on the device: always run the merge pass
    c->step_max_chunks =
        row_chunks(c->cfg.max_pages_per_seq, row_item_pages(c->dev_item_pages, batch, batch), c->dev_chunk_cap);
    c->step_batch = batch;
    c->step_entries = c->dev_entries_cap;
    c->page_stride = c->dev_stride;
    return KVC_OK;
}

int kv_cache_sync(kv_cache* c)
{
    if (!c) return fail(KVC_ERR_INVALID, "kv_cache_sync: null cache");
    if (c->host_only) return KVC_OK;
    return sync_from_device(c);
}

int kv_selftest_wait_timeout(int64_t limit_ns, int32_t* status, void* stream)
{
    if (!status || limit_ns <= 0 || limit_ns > 2000000000ll)
        return fail(KVC_ERR_INVALID, "kv_selftest_wait_timeout: status must be non-null, 0 < limit_ns <= 2e9");
    KVD_CUDA(launch_wait_timeout_check((uint64_t)limit_ns, status, static_cast<cudaStream_t>(stream)));
    return KVC_OK;
}

}  // extern "C"
