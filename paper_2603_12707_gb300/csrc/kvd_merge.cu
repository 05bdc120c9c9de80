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

// Merge pass.  SPLIT warps merge a split row's items for one query head
// h = g * G + hh of batch row b, each owning D / SPLIT dims:
//     M = max_c m_c,  O = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c,
// lane c holding the (m, l) of item c (and, in the 32-item variant, of item
// c + 32: rows of up to 64 items) and every lane D / (32 * SPLIT) dims of o.  The loads of (m, l) and of the first BATCH items' o are
// issued before the first use, so a row of up to BATCH items costs one round
// trip to L2.
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
    // Only the 32-item variant takes rows of more than 32 items; the smaller
    // variants keep their registers (they must fit beside the split pass).
    constexpr bool kTwoSlots = BATCH == 32;
    float2 ml0 = make_float2(-INFINITY, 0.f), ml1 = make_float2(-INFINITY, 0.f);
    if (lane < nch) ml0 = __ldcg(&p.part_ml[slot(lane)]);
    if constexpr (kTwoSlots)
        if (lane + 32 < nch) ml1 = __ldcg(&p.part_ml[slot(lane + 32)]);
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
    float M = kTwoSlots ? fmaxf(ml0.x, ml1.x) : ml0.x;
#pragma unroll
    for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    // Items lane and lane + 32 weigh e = 2^(m - M); the sum of e * o is
    // divided by L = sum e * l at the end, so the reduction of L runs beside
    // the weighted sum instead of before it.
    const float e0 = (lane < nch) ? ex2(ml0.x - M) : 0.f;
    const float e1 = (kTwoSlots && lane + 32 < nch) ? ex2(ml1.x - M) : 0.f;
    float L = kTwoSlots ? e0 * ml0.y + e1 * ml1.y : e0 * ml0.y;
#pragma unroll
    for (int o = 16; o; o >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o);
    float acc[PER];
#pragma unroll
    for (int j = 0; j < PER; ++j) acc[j] = 0.f;
    for (int c0 = 0; c0 < nch; c0 += BATCH) {
        if (c0) load(c0);
#pragma unroll
        for (int u = 0; u < BATCH; ++u) {
            const float wc = __shfl_sync(0xffffffffu, (!kTwoSlots || c0 + u < 32) ? e0 : e1, (c0 + u) & 31);
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

// The smallest variant whose items in flight cover the step's longest row,
// unless its registers would leave part of the grid waiting for a slot beside
// the resident split pass: then fewer items in flight (a second round trip
// for the longest rows only) with fewer registers.
cudaError_t launch_merge(int D, bool pdl, int max_chunks, int num_sms, int split_regs_per_subpartition,
                         const DecodeParams& p, cudaStream_t st)
{
    const int64_t units = (int64_t)p.batch * p.H_q * kMergeSplit;
    const int64_t want = std::max<int64_t>(1, std::min<int64_t>((units + kMergeWarps - 1) / kMergeWarps,
                                                                  (int64_t)num_sms * kMergeGridPerSm));
    int batch = max_chunks <= 4 ? 4 : max_chunks <= 8 ? 8 : max_chunks <= 16 ? 16 : 32;
    int64_t grid = want;
    // Rows of more than 32 items need the 32-item variant (two (m, l) per lane).
    const int min_batch = max_chunks > 32 ? 32 : 4;
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
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kMergeWarps * 32);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    const int flag = pdl ? 1 : 0;
    if (D == 128) return launch_merge_d<128>(batch, cfg, p, flag);
    if (D == 64) return launch_merge_d<64>(batch, cfg, p, flag);
    return cudaErrorInvalidValue;
}

}  // namespace kvd
