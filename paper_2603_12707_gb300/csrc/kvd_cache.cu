// Page-table maintenance, the per-step update and split plan, token writes /
// reads into pages, and the fused K+V append (kv_append).
#include <algorithm>
#include <climits>

#include "kvd_internal.h"
#include "kvd_ptx.cuh"

namespace kvd {

namespace {

__device__ __forceinline__ void flag_error(int32_t* err, int bit) { atomicOr(err, bit); }

__global__ void scatter_i32_kernel(int32_t* base, const __grid_constant__ ScatterI32 s)
{
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < s.n; i += gridDim.x * blockDim.x)
        base[s.idx[i]] = s.val[i];
}

// Exclusive block-wide prefix sum of one int per thread (blockDim.x = 1024).
__device__ int block_exclusive_scan(int v, int* total)
{
    __shared__ int warp_sums[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = (lane < (int)(blockDim.x >> 5)) ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        warp_sums[lane] = w;   // inclusive over warps
    }
    __syncthreads();
    const int before_warp = warp ? warp_sums[warp - 1] : 0;
    *total = warp_sums[31];
    __syncthreads();
    return before_warp + x - v;
}

// Split plan of a step, built by one block of 1024 threads: plan position i
// takes batch row b, sequence seq, len tokens from row_at(i, &b, &seq, &len);
// the row is cut into row_chunks() items of near-equal size, a row's items
// adjacent, its target size graduated by position (row_item_pages).  Entries
// past max_entries are dropped with error bit 4.  Each entry's page ids are
// copied from the page table into pages_out (stride page_stride), so the
// decode kernel reads them alongside the entry.  Returns the entries planned.
template <class RowAt>
__device__ int build_split_plan(int batch, int item_pages, int chunk_cap, int max_entries, RowAt row_at,
                                PlanEntry* plan, int2* rows, const int32_t* page_table, int max_pages,
                                int32_t* pages_out, int page_stride, int32_t* err)
{
    __shared__ int s_seq[1024], s_np[1024], s_off[1024], s_nch[1024];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int carry = 0;
    for (int base = 0; base < batch; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int b = 0, seq = 0, len = 0, np = 0, nch = 0;
        if (i < batch) {
            row_at(i, &b, &seq, &len);
            np = (len + kPageSize - 1) / kPageSize;
            nch = row_chunks(np, row_item_pages(item_pages, i, batch), chunk_cap);
        }
        int total;
        const int off = carry + block_exclusive_scan(nch, &total);
        if (off + nch > max_entries) {
            flag_error(err, 4);
            nch = 0;
        }
        for (int c = 0; c < nch; ++c) {
            int first, n;
            chunk_range(np, nch, c, &first, &n);
            plan[off + c] = PlanEntry{b, seq, len, first, n, c, nch, off};
        }
        if (i < batch) rows[b] = make_int2(off, nch);
        s_seq[threadIdx.x] = seq;
        s_np[threadIdx.x] = np;
        s_off[threadIdx.x] = off;
        s_nch[threadIdx.x] = nch;
        __syncthreads();
        // Page ids: each row gets (warps / rows) warps, at least one; a warp
        // copies 32-page windows of its row, four windows in flight per lane.
        // Page j of a row lies in item c at offset o (chunk_range inverted:
        // the first np % nch items hold one page more).
        const int n_rows = min((int)blockDim.x, batch - base);
        const int n_warps = (int)(blockDim.x >> 5);
        const int per_row = n_rows >= n_warps ? 1 : n_warps / n_rows;
        for (int t = warp; t < n_rows * per_row; t += n_warps) {
            const int r = t / per_row, part = t - r * per_row;
            const int rnp = s_np[r], rnch = s_nch[r];
            if (rnch == 0) continue;
            const int small = rnp / rnch, extra = rnp % rnch, big_pages = extra * (small + 1);
            const int32_t* src = page_table + (int64_t)s_seq[r] * max_pages;
            for (int w0 = part; w0 * 32 < rnp; w0 += 4 * per_row) {
                int32_t v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int j = (w0 + u * per_row) * 32 + lane;
                    v[u] = j < rnp ? src[j] : 0;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int j = (w0 + u * per_row) * 32 + lane;
                    if (j >= rnp) continue;
                    int c, o;
                    if (j < big_pages) {
                        c = j / (small + 1);
                        o = j - c * (small + 1);
                    } else {
                        c = extra + (j - big_pages) / small;
                        o = j - big_pages - (c - extra) * small;
                    }
                    if (o < page_stride)
                        pages_out[(int64_t)(s_off[r] + c) * page_stride + o] = v[u];
                    else
                        flag_error(err, 4);
                }
            }
        }
        __syncthreads();   // the next chunk of rows reuses the shared arrays
        carry += total;
    }
    return carry;
}

// Apply the step's length / page-table updates; in the last launch of a step,
// build the split plan with the rows in the host's order (longest first when
// the batch fits one launch).  The host sized the plan for exactly this step.
__global__ void __launch_bounds__(1024)
    step_kernel(const __grid_constant__ StepPatch patch, const __grid_constant__ PlanArgs a)
{
    for (int i = threadIdx.x; i < patch.n; i += blockDim.x) {
        const int seq = patch.seq[i], len = patch.new_len[i];
        a.seq_len[seq] = len;
        a.step_seq[patch.b0 + i] = seq;
        if (patch.new_page[i] >= 0)
            a.page_table[(int64_t)seq * a.max_pages + (len - 1) / kPageSize] = patch.new_page[i];
    }
    if (!a.build) return;
    __syncthreads();
    build_split_plan(
        a.batch, a.item_pages, a.chunk_cap, INT_MAX,
        [&](int i, int* b, int* seq, int* len) {
            *b = a.use_order ? a.order[i] : i;
            *seq = a.step_seq[*b];
            *len = a.seq_len[*seq];
            if (*len <= 0 || *len > a.max_pages * kPageSize) {
                flag_error(a.err, 4);
                *len = 1;
            }
        },
        a.plan, a.rows, a.page_table, a.max_pages, a.page_ids, a.page_stride, a.err);
    if (threadIdx.x == 0) *a.step_no += 1u;
}

// The same step on the device (graph-replayable, no host input): rows in
// batch order reserve position len; a row whose position opens a page takes
// the next page of the device free stack, in batch order (the same pages the
// host allocator would hand out); then the split plan, rows longest first
// (stable, as on the host) when the batch fits one block, else in batch order.
// A row whose step fails (a sequence id outside [0, max_seqs), a full page
// row, or an exhausted pool: error bits 4 / 8) keeps its length and gets
// step_seq -1 and no work items, so the layer calls that follow neither write
// its cache nor its output row.  With the batch in one block, each row's
// sequence and new length stay in shared memory for the ranking and the plan.
__global__ void __launch_bounds__(1024) step_device_kernel(const StepDevArgs a)
{
    __shared__ int s_top;
    __shared__ int s_seq[1024], s_len[1024];   // per batch row when the batch fits the block
    const bool small = a.batch <= (int)blockDim.x;
    if (threadIdx.x == 0) s_top = *a.free_top;
    int top0 = 0;
    int carry = 0;
    for (int base = 0; base < a.batch; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int seq = -1, len = 0, need = 0;
        bool ok = false;
        if (i < a.batch) {
            seq = a.seq_ids[i];
            if (seq >= 0 && seq < a.max_seqs) {
                len = a.seq_len[seq];
                ok = len >= 0 && len + 1 <= a.max_pages * kPageSize;
            }
            if (!ok) flag_error(a.err, 4);
            need = (ok && len % kPageSize == 0) ? 1 : 0;
        }
        int total;
        const int rank = carry + block_exclusive_scan(need, &total);   // also orders s_top's write
        if (base == 0) top0 = s_top;
        if (ok) {
            int32_t page = -1;
            if (need) {
                const int idx = top0 - 1 - rank;
                if (idx < 0) {
                    flag_error(a.err, 8);   // pool exhausted
                    ok = false;
                } else {
                    page = a.free_pages[idx];
                }
            }
            if (ok) {
                if (page >= 0) a.page_table[(int64_t)seq * a.max_pages + len / kPageSize] = page;
                a.seq_len[seq] = len + 1;
                len += 1;
            }
        }
        if (i < a.batch) {
            a.step_seq[i] = ok ? seq : -1;
            if (small) {
                s_seq[i] = ok ? seq : -1;
                s_len[i] = ok ? len : 0;
            }
        }
        carry += total;
    }
    __syncthreads();
    if (threadIdx.x == 0) *a.free_top = top0 - min(carry, top0);

    // Row order: the rank of row b counts the rows with more pages, and the
    // rows with as many pages that come before b (failed rows have none).
    __shared__ int s_np[1024];
    __shared__ int s_order[1024];
    if (small) {
        const int b = threadIdx.x;
        int np = 0;
        if (b < a.batch) {
            np = (s_len[b] + kPageSize - 1) / kPageSize;
            s_np[b] = np;
        }
        __syncthreads();
        if (b < a.batch) {
            int rank = 0;
            for (int j = 0; j < a.batch; ++j) {
                const int o = s_np[j];
                rank += (o > np || (o == np && j < b)) ? 1 : 0;
            }
            s_order[rank] = b;
        }
        __syncthreads();
    }
    const int entries = build_split_plan(
        a.batch, a.item_pages, a.chunk_cap, a.max_entries,
        [&](int i, int* b, int* seq, int* len) {
            *b = small ? s_order[i] : i;
            *seq = small ? s_seq[*b] : a.step_seq[*b];
            *len = *seq < 0 ? 0 : (small ? s_len[*b] : a.seq_len[*seq]);   // 0 tokens: no items
            if (*seq < 0) *seq = 0;
        },
        a.plan, a.rows, a.page_table, a.max_pages, a.page_ids, a.page_stride, a.err);
    if (threadIdx.x == 0) {
        *a.n_entries = min(entries, a.max_entries);
        *a.step_no += 1u;
    }
}

// Reserve n tokens for a sequence, or release all its pages, on the device
// free stack, in stream order with device-side steps: a reservation takes
// the next pages of the stack for the logical pages its new positions open
// (all or nothing: a full page row sets bit 4, an exhausted pool bit 8, and
// nothing changes); a release puts the pages back on top of the stack so that
// its logical page 0 is handed out next, clears its page-table row and sets
// its length to 0.
__global__ void __launch_bounds__(256) seq_op_kernel(const SeqOpArgs a)
{
    __shared__ int s_len, s_top, s_first, s_count;
    if (threadIdx.x == 0) {
        const int len = a.seq_len[a.seq];
        const int top = *a.free_top;
        int first = 0, count = 0;
        if (len < 0 || len > a.max_pages * kPageSize) {
            flag_error(a.err, 4);
        } else if (a.free_seq) {
            count = (len + kPageSize - 1) / kPageSize;
        } else {
            const int64_t end = (int64_t)len + a.n;
            first = (len + kPageSize - 1) / kPageSize;
            const int64_t need_total = (end + kPageSize - 1) / kPageSize;
            if (need_total > a.max_pages) {
                flag_error(a.err, 4);
            } else if (need_total - first > top) {
                flag_error(a.err, 8);
            } else {
                count = (int)(need_total - first);
                a.seq_len[a.seq] = (int)end;
            }
        }
        s_len = len;
        s_top = top;
        s_first = first;
        s_count = count;
    }
    __syncthreads();
    int32_t* row = a.page_table + (int64_t)a.seq * a.max_pages;
    const int top = s_top, first = s_first, count = s_count;
    if (a.free_seq) {
        for (int k = threadIdx.x; k < count; k += blockDim.x) {
            a.free_pages[top + count - 1 - k] = row[k];
            row[k] = -1;
        }
        if (threadIdx.x == 0 && s_len >= 0 && s_len <= a.max_pages * kPageSize) {
            *a.free_top = top + count;
            a.seq_len[a.seq] = 0;
        }
    } else {
        for (int k = threadIdx.x; k < count; k += blockDim.x) row[first + k] = a.free_pages[top - 1 - k];
        if (threadIdx.x == 0) *a.free_top = top - count;
    }
}

// One thread per 16-byte chunk of a [n][H_kv][D] token block.
__global__ void token_copy_kernel(const TokenCopyArgs a)
{
    if (a.len && a.first_pos + a.n > *a.len) {   // positions past the sequence's length
        if (blockIdx.x == 0 && threadIdx.x == 0) flag_error(a.err, 4);
        return;
    }
    const int chunks = a.D / 8;
    const int64_t total = (int64_t)a.n * a.H_kv * chunks;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % chunks);
        const int64_t tg = i / chunks;
        const int g = (int)(tg % a.H_kv);
        const int t = (int)(tg / a.H_kv);
        const int pos = a.first_pos + t;
        const int32_t page = a.pt_row[pos / kPageSize];
        if (page < 0 || page >= a.num_pages) {
            flag_error(a.err, 1);
            continue;
        }
        const int64_t poff = (((int64_t)page * a.H_kv + g) * kPageSize + pos % kPageSize) * a.D + c * 8;
        const int64_t toff = i * 8;
        if (a.to_pool) {
            *reinterpret_cast<uint4*>(a.pool_k + poff) = *reinterpret_cast<const uint4*>(a.tok_k + toff);
            *reinterpret_cast<uint4*>(a.pool_v + poff) = *reinterpret_cast<const uint4*>(a.tok_v + toff);
        } else {
            *reinterpret_cast<uint4*>(a.tok_k + toff) = *reinterpret_cast<const uint4*>(a.pool_k + poff);
            *reinterpret_cast<uint4*>(a.tok_v + toff) = *reinterpret_cast<const uint4*>(a.pool_v + poff);
        }
    }
}

// Bulk write of packed token blocks.  CTA x finds its block by a binary
// search over tile_start, reads the tile's page id once, then its threads
// stream the tile in the page's order ([H_kv][slot][D], 16-byte chunks, four
// per thread in flight) with streaming loads and stores: the source is read
// once and the pages are not read back soon.
constexpr int kVarlenThreads = 256;
constexpr int kVarlenUnroll = 4;

__global__ void __launch_bounds__(kVarlenThreads) varlen_write_kernel(const __grid_constant__ VarlenWriteArgs a)
{
    const int tile = blockIdx.x;
    int lo = 0, hi = a.n_blocks - 1;   // the last block with tile_start <= tile
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (a.tile_start[mid] <= tile) lo = mid;
        else hi = mid - 1;
    }
    const int first = a.first_pos[lo];
    const int page_idx = first / kPageSize + (tile - a.tile_start[lo]);
    const int p0 = max(first, page_idx * kPageSize);
    const int p1 = min(first + a.n_tok[lo], (page_idx + 1) * kPageSize);
    const int nt = p1 - p0;
    // A block that passes its sequence's length is refused whole (every tile
    // checks the block's end, not its own).
    if (a.seq_len && first + a.n_tok[lo] > a.seq_len[a.seq[lo]]) {
        if (threadIdx.x == 0) flag_error(a.err, 4);
        return;
    }
    const int32_t pid = a.page_table[(int64_t)a.seq[lo] * a.max_pages + page_idx];
    if (pid < 0 || pid >= a.num_pages) {
        if (threadIdx.x == 0) flag_error(a.err, 1);
        return;
    }
    const int cpr = a.D / 8;   // 16-byte chunks per (token, head) row
    const int total = a.H_kv * nt * cpr;
    const int64_t layer = blockIdx.y;
    const uint4* sk = reinterpret_cast<const uint4*>(a.k + layer * a.src_layer_stride);
    const uint4* sv = reinterpret_cast<const uint4*>(a.v + layer * a.src_layer_stride);
    uint4* dk = reinterpret_cast<uint4*>(a.pool_k + layer * a.pool_layer_stride) +
                (int64_t)pid * a.H_kv * kPageSize * cpr;
    uint4* dv = reinterpret_cast<uint4*>(a.pool_v + layer * a.pool_layer_stride) +
                (int64_t)pid * a.H_kv * kPageSize * cpr;
    const int64_t tok0 = (int64_t)a.src_row[lo] + (p0 - first);
    const int slot0 = p0 - page_idx * kPageSize;
    for (int base = threadIdx.x; base < total; base += kVarlenUnroll * kVarlenThreads) {
        uint4 rk[kVarlenUnroll], rv[kVarlenUnroll];
        int64_t doff[kVarlenUnroll];
#pragma unroll
        for (int u = 0; u < kVarlenUnroll; ++u) {
            const int idx = base + u * kVarlenThreads;
            if (idx < total) {
                const int c = idx % cpr;
                const int r = idx / cpr;
                const int h = r / nt;
                const int t = r - h * nt;
                const int64_t soff = ((tok0 + t) * a.H_kv + h) * cpr + c;
                doff[u] = ((int64_t)h * kPageSize + slot0 + t) * cpr + c;
                rk[u] = __ldcs(sk + soff);
                rv[u] = __ldcs(sv + soff);
            }
        }
#pragma unroll
        for (int u = 0; u < kVarlenUnroll; ++u) {
            if (base + u * kVarlenThreads < total) {
                __stcs(dk + doff[u], rk[u]);
                __stcs(dv + doff[u], rv[u]);
            }
        }
    }
}

// kv_append: one thread per 16-byte chunk of k_new / v_new ([B][H_kv][D]);
// the chunk goes to slot (len-1) % P of page page_table[seq][(len-1) / P].
__global__ void append_kernel(const AppendArgs a)
{
    const int chunks = a.D / 8;
    const int total = a.batch * a.H_kv * chunks;
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= total) return;
    const int c = i % chunks;
    const int bg = i / chunks;
    const int g = bg % a.H_kv;
    const int b = bg / a.H_kv;
    const int seq = a.step_seq[b];
    if (seq < 0) return;   // the row's device-side step failed (already flagged)
    const int pos = a.seq_len[seq] - 1;
    if (pos < 0 || pos >= a.max_pages * kPageSize) {
        flag_error(a.err, 4);
        return;
    }
    const int32_t page = a.page_table[(int64_t)seq * a.max_pages + pos / kPageSize];
    if (page < 0 || page >= a.num_pages) {
        flag_error(a.err, 1);
        return;
    }
    const int64_t poff = (((int64_t)page * a.H_kv + g) * kPageSize + pos % kPageSize) * a.D + c * 8;
    const int64_t noff = (int64_t)i * 8;
    const uint4 kk = *reinterpret_cast<const uint4*>(a.k_new + noff);
    const uint4 vv = *reinterpret_cast<const uint4*>(a.v_new + noff);
    *reinterpret_cast<uint4*>(a.pool_k + poff) = kk;
    *reinterpret_cast<uint4*>(a.pool_v + poff) = vv;
}

// One warp per plan entry: its page ids, contiguous, at entry * stride.
__global__ void gather_pages_kernel(const PlanEntry* plan, int32_t entries, const int32_t* entries_dev,
                                    const int32_t* page_table, int32_t max_pages, int32_t* item_pages,
                                    int32_t stride)
{
    const int lane = threadIdx.x & 31;
    if (entries_dev) entries = min(entries, *entries_dev);
    const int warps = (gridDim.x * blockDim.x) >> 5;
    for (int e = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; e < entries; e += warps) {
        const PlanEntry en = plan[e];
        const int32_t* src = page_table + (int64_t)en.seq * max_pages + en.first_page;
        int32_t* dst = item_pages + (int64_t)e * stride;
        for (int i = lane; i < en.n_pages; i += 32) dst[i] = src[i];
    }
}

// One warp waits, with the decode kernel's bounded wait, on an mbarrier that
// nothing arrives on; status = 1 when the wait gave up, 0 if it completed.
__global__ void wait_timeout_kernel(uint64_t limit_ns, int32_t* status)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&bar), 1);
        fence_mbar_init();
    }
    __syncwarp();
    const bool done = mbar_wait_bounded(smem_addr(&bar), 0, limit_ns);
    if (threadIdx.x == 0) *status = __all_sync(0xffffffffu, done) ? 0 : 1;
    else (void)__all_sync(0xffffffffu, done);
}

}  // namespace

cudaError_t launch_wait_timeout_check(uint64_t limit_ns, int32_t* status, cudaStream_t st)
{
    wait_timeout_kernel<<<1, 32, 0, st>>>(limit_ns, status);
    return cudaGetLastError();
}

cudaError_t launch_gather_pages(const PlanEntry* plan, int32_t entries, const int32_t* entries_dev,
                                const int32_t* page_table, int32_t max_pages, int32_t* item_pages, int32_t stride,
                                int num_sms, cudaStream_t st)
{
    if (entries <= 0) return cudaSuccess;
    const int64_t want = ((int64_t)entries + 7) / 8;
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)num_sms * 8));
    gather_pages_kernel<<<grid, 256, 0, st>>>(plan, entries, entries_dev, page_table, max_pages, item_pages,
                                              stride);
    return cudaGetLastError();
}

cudaError_t launch_seq_op(const SeqOpArgs& a, cudaStream_t st)
{
    seq_op_kernel<<<1, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_step_device(const StepDevArgs& a, cudaStream_t st)
{
    step_device_kernel<<<1, 1024, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_scatter_i32(int32_t* base, const ScatterI32& s, cudaStream_t st)
{
    if (s.n <= 0) return cudaSuccess;
    scatter_i32_kernel<<<(s.n + 255) / 256, 256, 0, st>>>(base, s);
    return cudaGetLastError();
}

cudaError_t launch_step(const StepPatch& patch, const PlanArgs& plan, cudaStream_t st)
{
    step_kernel<<<1, 1024, 0, st>>>(patch, plan);
    return cudaGetLastError();
}

cudaError_t launch_token_copy(const TokenCopyArgs& a, cudaStream_t st)
{
    const int64_t total = (int64_t)a.n * a.H_kv * (a.D / 8);
    if (total <= 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 65535) blocks = 65535;
    token_copy_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_varlen_write(const VarlenWriteArgs& a, int n_layers, cudaStream_t st)
{
    if (a.n_tiles <= 0 || n_layers <= 0) return cudaSuccess;
    varlen_write_kernel<<<dim3((unsigned)a.n_tiles, (unsigned)n_layers), kVarlenThreads, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_append(const AppendArgs& a, cudaStream_t st)
{
    const int total = a.batch * a.H_kv * (a.D / 8);
    if (total <= 0) return cudaSuccess;
    append_kernel<<<(total + 255) / 256, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace kvd
