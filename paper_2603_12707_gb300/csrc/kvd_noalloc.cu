// decode_attention_noalloc: decode attention over caller-owned paged K/V with
// no device allocation at all.
//
// Who needs it.  The kv_cache path allocates: its pools at creation and, when
// a step's split plan outgrows them, its plan and partial-result buffers with
// cudaMallocAsync.  Some callers may not allocate device memory while they
// serve: an engine plugin whose enqueue must run inside a memory budget fixed
// when the engine was built, a runtime whose device memory all belongs to
// another framework's allocator, or a latency-critical decode thread that must
// not take the allocator's locks.  Those callers own the K/V pools and page
// table themselves and call this entry point instead.
//
// Scratch.  The split plan, the per-item partial results, the per-row merge
// table and the work counters live in one file-scope __device__ array of
// kNoAllocScratchBytes (16 MiB) that every GPU loading this library holds
// until the process exits.  Host code cannot use the array's name as a device
// address; the first call on each device looks the address up with
// cudaGetSymbolAddress (make that first call before any stream capture) and
// later calls reuse it.  Every call shares the array and leaves its contents
// behind, so each call clears the counters it needs before use, and calls
// that overlap on the GPU (different streams, no ordering) race on it.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <string>

#include "kvd_internal.h"
#include "kvdecode.h"

namespace kvd {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;
constexpr int kNoAllocMaxBatch = 1024;

static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

struct NoAllocPlanArgs {
    int32_t batch;
    PlanEntry* plan;
    int2* rows;            // [batch]: (first partial slot, items)
    uint32_t* queue;
    int32_t* err;
    int32_t clear_err;
    // rows in planning order (longest first)
    int32_t row[kNoAllocMaxBatch];   // batch row
    int32_t len[kNoAllocMaxBatch];   // tokens attended
    int32_t off[kNoAllocMaxBatch];   // first plan entry of the row
    int32_t nch[kNoAllocMaxBatch];   // items of the row
    int32_t slot[kNoAllocMaxBatch];  // first partial slot (rows with one item use none)
};

// One block: clear the work counters, then write each row's items
// (near-equal page ranges) at the offsets the host computed.
__global__ void __launch_bounds__(1024) noalloc_plan_kernel(const __grid_constant__ NoAllocPlanArgs a)
{
    if (threadIdx.x == 0) {
        a.queue[0] = 0;
        if (a.clear_err) *a.err = 0;
    }
    for (int i = threadIdx.x; i < a.batch; i += blockDim.x) {
        const int np = (a.len[i] + kPageSize - 1) / kPageSize;
        for (int c = 0; c < a.nch[i]; ++c) {
            int first, n;
            chunk_range(np, a.nch[i], c, &first, &n);
            a.plan[a.off[i] + c] = PlanEntry{a.row[i], a.row[i], a.len[i], first, n, c, a.nch[i], a.slot[i]};
        }
        a.rows[a.row[i]] = make_int2(a.slot[i], a.nch[i]);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encoder()
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

// Device address of the scratch array on the current device, looked up once.
int scratch_address(uint8_t** out)
{
    static std::mutex mu;
    static uint8_t* addr[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess || dev < 0 || dev >= 64) {
        set_last_error((std::string("decode_attention_noalloc: cudaGetDevice: ") + cudaGetErrorString(e)).c_str());
        return KVC_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) {
            set_last_error(
                (std::string("decode_attention_noalloc: cudaGetSymbolAddress: ") + cudaGetErrorString(e)).c_str());
            return KVC_ERR_CUDA;
        }
        addr[dev] = static_cast<uint8_t*>(p);
    }
    *out = addr[dev];
    return KVC_OK;
}

size_t round256(size_t x) { return (x + 255) & ~size_t(255); }

int fail(int code, const char* msg)
{
    set_last_error((std::string("decode_attention_noalloc: ") + msg).c_str());
    return code;
}

}  // namespace
}  // namespace kvd

using namespace kvd;

extern "C" KVC_API int decode_attention_noalloc(const void* k_pool, const void* v_pool, int64_t num_pages,
                                                int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                                int32_t batch, const int32_t* page_table, int32_t max_pages,
                                                const int32_t* lens, const void* q, void* out,
                                                float softmax_scale, int32_t* device_error, void* stream)
{
    if (!k_pool || !v_pool || !page_table || !lens || !q || !out) return fail(KVC_ERR_INVALID, "null argument");
    const uintptr_t al = reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
                         reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(out);
    if (al & 15u) return fail(KVC_ERR_INVALID, "k_pool, v_pool, q and out must be 16-byte aligned");
    if (num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads)
        return fail(KVC_ERR_INVALID, "num_q_heads must be a positive multiple of num_kv_heads");
    const int G = num_q_heads / num_kv_heads;
    if (G > kMaxGroup) return fail(KVC_ERR_UNSUPPORTED, "more than 8 query heads per KV head");
    if (head_dim != 64 && head_dim != 128) return fail(KVC_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (batch < 1 || batch > kNoAllocMaxBatch) return fail(KVC_ERR_INVALID, "batch must be in 1 .. 1024");
    if (num_pages < 1 || num_pages * num_kv_heads * kPageSize >= (int64_t)1 << 31)
        return fail(KVC_ERR_INVALID, "num_pages must be >= 1 with num_pages * num_kv_heads * 16 < 2^31");
    if (max_pages < 1) return fail(KVC_ERR_INVALID, "max_pages must be >= 1");
    if (!(softmax_scale <= 0.f) && !std::isfinite(softmax_scale))
        return fail(KVC_ERR_INVALID, "softmax_scale must be finite");
    int64_t total_pages = 0;
    for (int b = 0; b < batch; ++b) {
        if (lens[b] < 1 || (int64_t)lens[b] > (int64_t)max_pages * kPageSize)
            return fail(KVC_ERR_INVALID, "every length must be in 1 .. max_pages * 16");
        total_pages += (lens[b] + kPageSize - 1) / kPageSize;
    }
    cudaStream_t st = static_cast<cudaStream_t>(stream);

    int dev = 0;
    DecodeVariant var{};
    int num_sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                  cudaSuccess)
        return fail(KVC_ERR_CUDA, "cannot query the current device");
    if (cudaError_t e = decode_variant_info(head_dim, G > 1, &var); e != cudaSuccess)
        return fail(KVC_ERR_CUDA, cudaGetErrorString(e));
    uint8_t* scratch = nullptr;
    if (int rc = scratch_address(&scratch)) return rc;

    // Items: the library's usual target (about three per resident warp),
    // enlarged until the plan and the partials fit the static scratch.
    const int64_t warps = (int64_t)num_sms * std::max(1, var.ctas_per_sm) * std::max(1, var.warps);
    int64_t T = std::min<int64_t>(128, std::max<int64_t>(2, (total_pages * num_kv_heads + 3 * warps - 1) / (3 * warps)));
    int64_t entries = 0;
    bool split_rows = false;
    int stride = 1;
    size_t off_pages = 0, off_o = 0, off_ml = 0, off_rows = 0, off_q = 0, off_err = 0, need = 0;
    // T doubles, clamped to kMaxItemPages; the attempt at kMaxItemPages is the last.
    for (;; T = std::min<int64_t>(2 * T, kMaxItemPages)) {
        entries = 0;
        int64_t split_items = 0;   // only rows cut into several items keep partials
        for (int b = 0; b < batch; ++b) {
            const int64_t nch = row_chunks((lens[b] + kPageSize - 1) / kPageSize, (int)T);
            entries += nch;
            if (nch > 1) split_items += nch;
        }
        split_rows = split_items > 0;
        const int64_t slots = split_items * num_kv_heads;
        stride = 1;
        for (int b = 0; b < batch; ++b) {
            const int np = (lens[b] + kPageSize - 1) / kPageSize;
            const int nch = row_chunks(np, (int)T);
            stride = std::max(stride, (np + nch - 1) / nch);
        }
        off_pages = round256((size_t)entries * sizeof(PlanEntry));
        off_o = round256(off_pages + (size_t)entries * stride * sizeof(int32_t));
        off_ml = round256(off_o + (size_t)slots * G * head_dim * sizeof(float));
        off_rows = round256(off_ml + (size_t)slots * G * sizeof(float2));
        off_q = round256(off_rows + (size_t)batch * sizeof(int2));
        off_err = off_q + 2 * sizeof(uint32_t);
        need = round256(off_err + sizeof(int32_t));
        if (need <= kNoAllocScratchBytes || T >= kMaxItemPages) break;
    }
    if (need > kNoAllocScratchBytes)
        return fail(KVC_ERR_UNSUPPORTED, ("the batch needs " + std::to_string(need) +
                                          " bytes of scratch; the static limit is 16 MiB").c_str());

    auto encode = encoder();
    if (!encode) return fail(KVC_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
    CUtensorMap maps[2];
    for (int kv = 0; kv < 2; ++kv) {
        CUresult r = encode_tile_map(reinterpret_cast<void*>(encode), &maps[kv], const_cast<void*>(kv ? v_pool : k_pool),
                                     num_pages * num_kv_heads * kPageSize, head_dim, 0);
        if (r != CUDA_SUCCESS) return fail(KVC_ERR_INVALID, "cuTensorMapEncodeTiled rejected the pools");
    }

    NoAllocPlanArgs pa;
    pa.batch = batch;
    pa.plan = reinterpret_cast<PlanEntry*>(scratch);
    pa.rows = reinterpret_cast<int2*>(scratch + off_rows);
    pa.queue = reinterpret_cast<uint32_t*>(scratch + off_q);
    pa.err = device_error ? device_error : reinterpret_cast<int32_t*>(scratch + off_err);
    pa.clear_err = device_error ? 0 : 1;
    {
        for (int b = 0; b < batch; ++b) pa.row[b] = b;
        std::stable_sort(pa.row, pa.row + batch, [&](int32_t x, int32_t y) { return lens[x] > lens[y]; });
        int32_t off = 0, slot = 0;
        for (int i = 0; i < batch; ++i) {
            const int32_t b = pa.row[i];
            const int32_t nch = row_chunks((lens[b] + kPageSize - 1) / kPageSize, (int)T);
            pa.len[i] = lens[b];
            pa.off[i] = off;
            pa.nch[i] = nch;
            pa.slot[i] = slot;
            off += nch;
            if (nch > 1) slot += nch;
        }
    }
    noalloc_plan_kernel<<<1, 1024, 0, st>>>(pa);
    if (cudaError_t e = cudaGetLastError(); e != cudaSuccess) return fail(KVC_ERR_CUDA, cudaGetErrorString(e));
    int32_t* item_pages = reinterpret_cast<int32_t*>(scratch + off_pages);
    if (cudaError_t e = launch_gather_pages(pa.plan, (int32_t)entries, nullptr, page_table, max_pages, item_pages, stride,
                                            num_sms, st);
        e != cudaSuccess)
        return fail(KVC_ERR_CUDA, cudaGetErrorString(e));

    const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt((float)head_dim);
    DecodeParams p;
    p.q = static_cast<const uint16_t*>(q);
    p.out = static_cast<uint16_t*>(out);
    p.page_table = page_table;
    p.plan = pa.plan;
    p.part_o = reinterpret_cast<float*>(scratch + off_o);
    p.part_ml = reinterpret_cast<float2*>(scratch + off_ml);
    p.rows = pa.rows;
    p.item_pages = item_pages;
    p.page_stride = stride;
    p.n_entries_dev = nullptr;
    p.batch = batch;
    p.queue = pa.queue;
    p.queue_next = nullptr;
    p.err = pa.err;
    p.num_pages = num_pages;
    p.n_items = (int32_t)(entries * num_kv_heads);
    p.H_kv = num_kv_heads;
    p.H_q = num_q_heads;
    p.G = G;
    p.max_pages = max_pages;
    p.scale_log2 = scale * 1.4426950408889634f;
    p.kv_map = 0;
    p.start_flags = nullptr;
    p.step_no = nullptr;
    p.tag = p.prev_tag = 0;
    p.num_sms = num_sms;
    p.k_new = p.v_new = nullptr;
    p.pool_k = p.pool_v = nullptr;
    const int64_t resident = (int64_t)num_sms * std::max(1, var.ctas_per_sm);
    const int64_t want = (p.n_items + var.warps - 1) / var.warps;
    const int grid = (int)std::max<int64_t>(1, std::min(resident, want));
    if (cudaError_t e = launch_decode(head_dim, G > 1, false, false, grid, maps[0], maps[1], p, st); e != cudaSuccess)
        return fail(KVC_ERR_CUDA, cudaGetErrorString(e));
    if (split_rows)
        if (cudaError_t e = launch_merge(head_dim, false, kChunkCap, num_sms, 0, p, st); e != cudaSuccess)
            return fail(KVC_ERR_CUDA, cudaGetErrorString(e));
    return KVC_OK;
}
