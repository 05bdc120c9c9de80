// Merge pass of split-KV decode attention (sm_103a): the log-sum-exp merge of
// the partials (o, m, l) that the split pass (kvd_decode.cu) leaves for rows
// cut into several work items.  For batch row b and query head h of KV head
// g, with item c's running max m_c (log2 units), sum l_c and unnormalised
// accumulator o_c:
//     M = max_c m_c,  O = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c.
#include <math.h>

#include <algorithm>

#include "kvd_internal.h"
#include "kvd_ptx.cuh"

namespace kvd {

namespace {

// Merge pass.  SPLIT warps merge a split row's items (at most 32; longer rows
// go to merge_wide_kernel) for one query head h = g * G + hh of batch row b,
// each owning D / SPLIT dims:
//     M = max_c m_c,  O = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c,
// lane c holding the (m, l) of item c and every lane D / (32 * SPLIT) dims of
// o.  The loads of (m, l) and of the first BATCH items' o are issued before
// the first use, so a row of up to BATCH items costs one round trip to L2.
constexpr int kMergeSplit = 1;   // warps per (row, query head)
constexpr int kMergeWarps = 1;   // warps per CTA: small CTAs fit beside the split pass's
// Merge CTAs per SM at most.  The whole merge grid must fit beside the
// resident split pass (8 one-warp CTAs per SM): a merge CTA that waits for a
// slot holds back the next layer, which may start only once every merge CTA
// has started.  Rows with more units than the grid loop over them.
constexpr int kMergeGridPerSm = 16;

// BATCH: items whose o is loaded before the first use (registers: BATCH * D / 32
// floats per lane); the launch picks the smallest BATCH that covers the step's
// items per row, so a unit is one round trip and the CTAs stay small.
template <int D, int BATCH>
__device__ __forceinline__ void merge_unit(const DecodeParams& p, int2 row, int b, int g, int hh, int part,
                                           int lane)
{
    constexpr int PER = D / (32 * kMergeSplit);
    static_assert(PER == 1 || PER == 2 || PER == 4, "dims per lane");
    const int nch = row.y;
    auto slot = [&](int c) { return ((int64_t)(row.x + c) * p.H_kv + g) * p.G + hh; };
    float2 ml0 = make_float2(-INFINITY, 0.f);
    if (lane < nch) ml0 = __ldcg(&p.part_ml[slot(lane)]);
    const int d0 = part * (D / kMergeSplit) + lane * PER;
    float vals[BATCH][PER];
    auto load = [&](int c0) {
#pragma unroll
    for (int u = 0; u < BATCH; ++u) {
        const int c = c0 + u;
        const float* src = p.part_o + slot(c < nch ? c : 0) * D + d0;
        if (c < nch) {
            if constexpr (PER == 4) {
                const float4 t = __ldcg(reinterpret_cast<const float4*>(src));
                vals[u][0] = t.x; vals[u][1] = t.y; vals[u][2] = t.z; vals[u][3] = t.w;
            } else if constexpr (PER == 2) {
                const float2 t = __ldcg(reinterpret_cast<const float2*>(src));
                vals[u][0] = t.x; vals[u][1] = t.y;
            } else {
                vals[u][0] = __ldcg(src);
            }
        } else {
#pragma unroll
            for (int j = 0; j < PER; ++j) vals[u][j] = 0.f;
        }
    }
    };
    load(0);
    float M = ml0.x;
#pragma unroll
    for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    // Item lane weighs e = 2^(m - M); the sum of e * o is divided by
    // L = sum e * l at the end, so the reduction of L runs beside the
    // weighted sum instead of before it.
    const float e0 = (lane < nch) ? ex2(ml0.x - M) : 0.f;
    float L = e0 * ml0.y;
#pragma unroll
    for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
    float acc[PER];
#pragma unroll
    for (int j = 0; j < PER; ++j) acc[j] = 0.f;
    for (int c0 = 0; c0 < nch; c0 += BATCH) {
        if (c0) load(c0);
#pragma unroll
        for (int u = 0; u < BATCH; ++u) {
            const float wc = __shfl_sync(0xffffffffu, e0, (c0 + u) & 31);
#pragma unroll
            for (int j = 0; j < PER; ++j) acc[j] = fmaf(wc, vals[u][j], acc[j]);
        }
    }
    const float inv = 1.f / L;
#pragma unroll
    for (int j = 0; j < PER; ++j) acc[j] *= inv;
    uint16_t* orow = p.out + ((int64_t)b * p.H_q + g * p.G + hh) * D + d0;
    if constexpr (PER == 4) {
        *reinterpret_cast<uint2*>(orow) = make_uint2(pack_bf16(acc[0], acc[1]), pack_bf16(acc[2], acc[3]));
    } else if constexpr (PER == 2) {
        *reinterpret_cast<uint32_t*>(orow) = pack_bf16(acc[0], acc[1]);
    } else {
        orow[0] = (uint16_t)(pack_bf16(acc[0], 0.f) & 0xffffu);
    }
}

// Second pass: kMergeSplit warps per (row, query head) of a split row.  The
// row descriptors come from the step's plan, not from the split pass, so a
// warp reads its first one before waiting for the split pass: after the
// wait only the partials are fetched.
template <int D, int BATCH>
__global__ void __launch_bounds__(kMergeWarps * 32) merge_kernel(const DecodeParams p, int pdl)
{
    const int lane = threadIdx.x & 31;
    const int total = p.batch * p.H_q * kMergeSplit;
    int w = blockIdx.x * kMergeWarps + (threadIdx.x >> 5);
    int2 row = make_int2(0, 0);
    if (w < total) row = p.rows[(w / kMergeSplit) / p.H_q];
    if (pdl) {
        griddep_launch_dependents();   // the next layer may start streaming now
        griddep_wait();                // the split pass of this layer is complete
    }
    // Announce that the split pass is complete to the next layer's warps,
    // which are resident already and warm L2 while this pass runs.
    if (blockIdx.x == 0 && p.start_flags) {
        const uint32_t v = *p.step_no * 65536u + p.tag;
        for (int k = lane; k < p.num_sms; k += 32) p.start_flags[k * 32] = v;
    }
    for (bool first = true; w < total; w += gridDim.x * kMergeWarps, first = false) {
        const int part = w % kMergeSplit;
        const int bh = w / kMergeSplit;
        const int b = bh / p.H_q, h = bh - b * p.H_q;
        if (!first) row = p.rows[b];
        if (row.y <= 1) continue;
        const int g = h / p.G;
        merge_unit<D, BATCH>(p, row, b, g, h - g * p.G, part, lane);
    }
}

// Rows of more than 32 items (at most 64): one CTA of four warps per (row,
// query head).  Warp w merges items 16w .. 16w+15 in one round trip to L2,
//     M_w = max_c m_c,  L_w = sum_c 2^(m_c - M_w) l_c,  O_w = sum_c 2^(m_c - M_w) o_c,
// and the four results combine in shared memory:
//     M = max_w M_w,  O = sum_w 2^(M_w - M) O_w / sum_w 2^(M_w - M) L_w,
// the same log-sum-exp merge, regrouped (a warp with no items has M_w = -inf
// and weighs 0), in one round trip where a single warp would need two.
constexpr int kWideWarps = 4;
constexpr int kWideItems = 16;   // items per warp
static_assert(kWideWarps * kWideItems >= kMaxChunks, "a row's items (at most kMaxChunks) fit one CTA");

template <int D>
__global__ void __launch_bounds__(kWideWarps * 32) merge_wide_kernel(const DecodeParams p, int pdl)
{
    constexpr int PER = D / 32;
    __shared__ float s_o[kWideWarps][D];
    __shared__ float2 s_ml[kWideWarps];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int total = p.batch * p.H_q;
    int u = blockIdx.x;
    int2 row = make_int2(0, 0);
    if (u < total) row = p.rows[u / p.H_q];
    if (pdl) {
        griddep_launch_dependents();   // the next layer may start streaming now
        griddep_wait();                // the split pass of this layer is complete
    }
    if (blockIdx.x == 0 && wid == 0 && p.start_flags) {
        const uint32_t v = *p.step_no * 65536u + p.tag;
        for (int k = lane; k < p.num_sms; k += 32) p.start_flags[k * 32] = v;
    }
    for (bool first = true; u < total; u += gridDim.x, first = false) {
        const int b = u / p.H_q, h = u - b * p.H_q;
        if (!first) row = p.rows[b];
        if (row.y <= 1) continue;      // the same for every warp of the CTA
        const int g = h / p.G, hh = h - g * p.G;
        const int c0 = wid * kWideItems;
        const int n = max(0, min(kWideItems, row.y - c0));
        auto slot = [&](int c) { return ((int64_t)(row.x + c) * p.H_kv + g) * p.G + hh; };
        const float2 ml = lane < n ? __ldcg(&p.part_ml[slot(c0 + lane)]) : make_float2(-INFINITY, 0.f);
        // Every load goes out before the first use; a slot past the warp's
        // items reads the row's item 0 (a finite partial) and weighs 0.
        float vals[kWideItems][PER];
#pragma unroll
        for (int i = 0; i < kWideItems; ++i) {
            const float* src = p.part_o + slot(i < n ? c0 + i : 0) * D + lane * PER;
            if constexpr (PER == 4) {
                const float4 t = __ldcg(reinterpret_cast<const float4*>(src));
                vals[i][0] = t.x; vals[i][1] = t.y; vals[i][2] = t.z; vals[i][3] = t.w;
            } else {
                const float2 t = __ldcg(reinterpret_cast<const float2*>(src));
                vals[i][0] = t.x; vals[i][1] = t.y;
            }
        }
        float M = ml.x;
#pragma unroll
        for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
        const float e = lane < n ? ex2(ml.x - M) : 0.f;
        float L = e * ml.y;
#pragma unroll
        for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
        float acc[PER];
#pragma unroll
        for (int j = 0; j < PER; ++j) acc[j] = 0.f;
        // (a loop of n / 16 rounded up: once, or not at all; its runtime bound
        // keeps every load above ahead of the first multiply-add)
        for (int c = 0; c < n; c += kWideItems) {
#pragma unroll
            for (int i = 0; i < kWideItems; ++i) {
                const float w = __shfl_sync(0xffffffffu, e, i);
#pragma unroll
                for (int j = 0; j < PER; ++j) acc[j] = fmaf(w, vals[i][j], acc[j]);
            }
        }
        if (lane == 0) s_ml[wid] = make_float2(M, L);
#pragma unroll
        for (int j = 0; j < PER; ++j) s_o[wid][lane * PER + j] = acc[j];
        __syncthreads();
        if (wid == 0) {
            float Mx = s_ml[0].x;
#pragma unroll
            for (int w = 1; w < kWideWarps; ++w) Mx = fmaxf(Mx, s_ml[w].x);
            float Ls = 0.f, o[PER];
#pragma unroll
            for (int j = 0; j < PER; ++j) o[j] = 0.f;
#pragma unroll
            for (int w = 0; w < kWideWarps; ++w) {
                const float sw = ex2(s_ml[w].x - Mx);   // 0 for a warp without items
                Ls = fmaf(sw, s_ml[w].y, Ls);
#pragma unroll
                for (int j = 0; j < PER; ++j) o[j] = fmaf(sw, s_o[w][lane * PER + j], o[j]);
            }
            const float inv = 1.f / Ls;
            uint16_t* orow = p.out + ((int64_t)b * p.H_q + h) * D + lane * PER;
            if constexpr (PER == 4) {
                *reinterpret_cast<uint2*>(orow) = make_uint2(pack_bf16(o[0] * inv, o[1] * inv),
                                                             pack_bf16(o[2] * inv, o[3] * inv));
            } else {
                *reinterpret_cast<uint32_t*>(orow) = pack_bf16(o[0] * inv, o[1] * inv);
            }
        }
        __syncthreads();               // s_o and s_ml are reused by the next unit
    }
}

// The merge pass uses no shared memory; asking for the largest shared-memory
// carveout keeps an SM that hosts its CTAs in the configuration of the split
// pass, so the next layer's split-pass CTAs can still be placed there.
template <int D, int BATCH>
cudaError_t launch_merge_variant(const cudaLaunchConfig_t& cfg, const DecodeParams& p, int flag)
{
    static cudaError_t status =
        cudaFuncSetAttribute(merge_kernel<D, BATCH>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (status != cudaSuccess) return status;
    return cudaLaunchKernelEx(&cfg, merge_kernel<D, BATCH>, p, flag);
}

template <int D>
cudaError_t launch_merge_wide(const cudaLaunchConfig_t& cfg, const DecodeParams& p, int flag)
{
    static cudaError_t status =
        cudaFuncSetAttribute(merge_wide_kernel<D>, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (status != cudaSuccess) return status;
    return cudaLaunchKernelEx(&cfg, merge_wide_kernel<D>, p, flag);
}

template <int D>
int merge_wide_registers()
{
    static int regs = [] {
        cudaFuncAttributes a;
        return cudaFuncGetAttributes(&a, merge_wide_kernel<D>) == cudaSuccess ? a.numRegs : 255;
    }();
    return regs;
}

template <int D, int BATCH>
int merge_registers()
{
    static int regs = [] {
        cudaFuncAttributes a;
        return cudaFuncGetAttributes(&a, merge_kernel<D, BATCH>) == cudaSuccess ? a.numRegs : 255;
    }();
    return regs;
}

template <int D>
int merge_registers(int batch)
{
    return batch == 4 ? merge_registers<D, 4>() : batch == 8 ? merge_registers<D, 8>()
         : batch == 16 ? merge_registers<D, 16>() : merge_registers<D, 32>();
}

template <int D>
cudaError_t launch_merge_d(int batch, cudaLaunchConfig_t& cfg, const DecodeParams& p, int flag)
{
    if (batch == 4) return launch_merge_variant<D, 4>(cfg, p, flag);
    if (batch == 8) return launch_merge_variant<D, 8>(cfg, p, flag);
    if (batch == 16) return launch_merge_variant<D, 16>(cfg, p, flag);
    return launch_merge_variant<D, 32>(cfg, p, flag);
}

}  // namespace

// Rows of up to 32 items: the smallest variant whose items in flight cover
// the step's longest row, unless its registers would leave part of the grid
// waiting for a slot beside the resident split pass: then fewer items in
// flight (a second round trip for the longest rows only) with fewer
// registers.  Longer rows: merge_wide_kernel.
cudaError_t launch_merge(int D, bool pdl, int max_chunks, int num_sms, int split_regs_per_subpartition,
                         const DecodeParams& p, cudaStream_t st)
{
    const int64_t units = (int64_t)p.batch * p.H_q * kMergeSplit;
    cudaLaunchConfig_t cfg = {};
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const int flag = pdl ? 1 : 0;
    // Rows of more than 32 items: four-warp CTAs, one round trip (merge_wide_kernel);
    // as many CTAs as fit beside the resident split pass (a CTA puts one warp on
    // each scheduler), at least one per SM.
    if (max_chunks > 32) {
        if (D != 128 && D != 64) return cudaErrorInvalidValue;
        const int regs = D == 128 ? merge_wide_registers<128>() : merge_wide_registers<64>();
        const int64_t per_sub = (kRegistersPerSubpartition - split_regs_per_subpartition) /
                                warp_register_allocation(regs);
        const int64_t fit = (int64_t)num_sms * std::max<int64_t>(1, std::min<int64_t>(kMergeGridPerSm, per_sub));
        cfg.gridDim = dim3((unsigned)std::max<int64_t>(1, std::min(units, fit)));
        cfg.blockDim = dim3(kWideWarps * 32);
        return D == 128 ? launch_merge_wide<128>(cfg, p, flag) : launch_merge_wide<64>(cfg, p, flag);
    }
    const int64_t want = std::max<int64_t>(1, std::min<int64_t>((units + kMergeWarps - 1) / kMergeWarps,
                                                                  (int64_t)num_sms * kMergeGridPerSm));
    int batch = max_chunks <= 4 ? 4 : max_chunks <= 8 ? 8 : max_chunks <= 16 ? 16 : 32;
    int64_t grid = want;
    const int min_batch = 4;
    for (;; batch /= 2) {
        const int regs = D == 128 ? merge_registers<128>(batch) : merge_registers<64>(batch);
        const int64_t per_sub = (kRegistersPerSubpartition - split_regs_per_subpartition) /
                                (warp_register_allocation(regs) * kMergeWarps);
        const int64_t fit = (int64_t)num_sms * std::min<int64_t>(kMergeGridPerSm, 4 * per_sub);
        if (fit >= want || batch == min_batch) {
            grid = std::max<int64_t>(1, std::min(want, fit));
            break;
        }
    }
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kMergeWarps * 32);
    if (D == 128) return launch_merge_d<128>(batch, cfg, p, flag);
    if (D == 64) return launch_merge_d<64>(batch, cfg, p, flag);
    return cudaErrorInvalidValue;
}

}  // namespace kvd
