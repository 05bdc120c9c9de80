// Split-KV decode attention over the paged bf16 KV cache (sm_103a).
//
// Schedule.  A step's plan cuts every (sequence, KV head) into work items of
// consecutive pages.  A persistent grid of warps pulls items from a global
// counter; each warp runs its items independently:
//   * one lane streams the (page, head) tiles of K and V into the warp's
//     private ring of R shared-memory stages, one 4-D TMA tile load per page
//     covering K and V (128-byte swizzle, L2 evict-first), completing on one
//     mbarrier per stage;
//   * the warp computes an online softmax over the item's tokens for the G
//     query heads of the KV head (reference max m in log2 units, running sum
//     l = sum 2^(s - m), unnormalised accumulator o, all fp32; m trails the
//     running max by at most 8, so most pages skip the rescale);
//   * a row with one item writes bf16 output directly; otherwise each item
//     stores (o, m, l) as a partial and a second pass (merge_kernel in
//     kvd_merge.cu: one warp per (row, query head), one lane per item's
//     (m, l), every item's o in flight at once) merges them by log-sum-exp:
//         M = max_c m_c,  O = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c.
// MHA (G = 1, 1 flop per byte) runs on the CUDA cores; GQA (2 <= G <= 8) runs
// Q.K^T and P.V as m16n8k16 bf16 MMAs with the 16 tokens of a page as M and the
// G heads (padded to 8) as N.
//
// Chained launches (programmatic dependent launch, decode_attention_append
// after another attention launch): a warp issues its first item's ring loads
// before the dependency wait; once the previous launch's merge pass announces
// (start_flags) that its split pass is complete, the warp brings the item's
// next kEarlyL2Pages pages into L2; and right after its wait it brings the
// next kRampL2Pages, so the HBM keeps streaming while the merge runs and the
// ring's pages are worked.  Consecutive launches use alternating work counters; each
// launch resets the next one's after its wait, so no warp does an atomic on
// its way out.
//
// Every mbarrier wait is bounded: after a second without progress the warp
// records KVC_DEVERR_WAIT_TIMEOUT, waits (bounded) for its loads in flight and
// leaves.  Page ids outside the pool are recorded and replaced by page 0.
// Device code only (included by kvd_decode.cu, which instantiates and
// launches it).
#pragma once

#include <math.h>

#include <type_traits>

#include "kvd_internal.h"
#include "kvd_ptx.cuh"

namespace kvd {

namespace {

constexpr uint64_t kWaitLimitNs = 1000000000ull;
// Pages of a warp's first item brought into L2 when its dependency wait
// returns, beyond the ring's stages: the HBM gets new requests at once
// instead of after the first page's work (Qwen-shaped layers +4 %, the long
// context +3 %; 1 or 3-4 pages measured no better).
constexpr int kRampL2Pages = 2;
// Pages brought into L2 earlier still, once the previous launch's merge pass
// has announced that its split pass is complete (while that merge runs):
// +0.4 % per step on the LLaVA and Qwen shapes; 2-3 pages cost the Qwen shape.
constexpr int kEarlyL2Pages = 1;
// How long a warp waits for that announcement at most (it comes once the
// previous split pass has ended, which chained CTAs see from its tail; the
// dependency wait follows in any case).
constexpr uint64_t kEarlyPollLimitNs = 500000ull;
constexpr int kWarps = 1;   // one warp per CTA: a CTA's resources free up as soon as its warp is done

template <int D, bool GQA>
struct Geo {
    static constexpr int kTileBytes = kPageSize * D * 2; // one (page, head) tile
    static constexpr int kStageBytes = 2 * kTileBytes;   // K tile + V tile
    // stages per warp (8 one-warp CTAs per SM at d = 128); deeper rings with
    // fewer warps, and for GQA a 2-stage ring with 12 warps, measured slower
    static constexpr int kRing = D == 128 ? 3 : 6;
    static constexpr int kRingBytes = kWarps * kRing * kStageBytes;
    static constexpr int kSmem = kRingBytes + kWarps * kRing * 8 + 1024;
};

// Byte offset of 16-byte chunk c (0 .. D/8-1) of tile row r: TMA writes a
// tile as D/64 blocks of [16 rows][64 cols] (2 KiB each), 128-byte swizzle.
__device__ __forceinline__ uint32_t swz(int r, int c)
{
    return (uint32_t)((c >> 3) * 2048 + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

// q . k over one 16-byte chunk (8 dims): k bf16, q as four f32 pairs.
__device__ __forceinline__ float dot8(const uint4& k, const uint64_t (&q2)[4])
{
    uint64_t acc = f2_fma(q2[0], bf16x2_to_f2(k.x), 0ull);
    acc = f2_fma(q2[1], bf16x2_to_f2(k.y), acc);
    acc = f2_fma(q2[2], bf16x2_to_f2(k.z), acc);
    acc = f2_fma(q2[3], bf16x2_to_f2(k.w), acc);
    float lo, hi;
    f2_unpack(acc, lo, hi);
    return lo + hi;
}

// o += p * v over one 16-byte chunk, o as four f32 pairs.
__device__ __forceinline__ void axpy8(uint64_t (&o2)[4], uint64_t p2, const uint4& v)
{
    o2[0] = f2_fma(p2, bf16x2_to_f2(v.x), o2[0]);
    o2[1] = f2_fma(p2, bf16x2_to_f2(v.y), o2[1]);
    o2[2] = f2_fma(p2, bf16x2_to_f2(v.z), o2[2]);
    o2[3] = f2_fma(p2, bf16x2_to_f2(v.w), o2[3]);
}

// ------------------------------------------------------------ MHA, CUDA cores
// A lane owns 16-byte chunk c of a row; TPI rows are covered per warp load.
template <int D>
struct MhaCompute {
    static constexpr int CH = D / 8;
    static constexpr int TPI = 32 / CH;
    static constexpr int IT = kPageSize / TPI;
    static constexpr int LOG_IT = (IT == 8) ? 3 : (IT == 4 ? 2 : 1);
    int c, tsub;
    uint64_t q2[4];          // q of this lane's chunk as f32 pairs
    float m, l;
    uint64_t o2[4];          // unnormalised output of this lane's chunk, f32 pairs

    __device__ __forceinline__ void start(const DecodeParams& p, const PlanEntry& en, int g, int lane)
    {
        c = lane % CH;
        tsub = lane / CH;
        const uint4 qq = *reinterpret_cast<const uint4*>(p.q + ((int64_t)en.b * p.H_q + g) * D + c * 8);
        q2[0] = bf16x2_to_f2(qq.x);
        q2[1] = bf16x2_to_f2(qq.y);
        q2[2] = bf16x2_to_f2(qq.z);
        q2[3] = bf16x2_to_f2(qq.w);
        m = -INFINITY;
        l = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) o2[k] = 0ull;
    }

    __device__ __forceinline__ void page(uint8_t* sK, uint8_t* sV, uint32_t, uint32_t, int valid,
                                         float scale_log2, int lane)
    {
        float part[IT];
#pragma unroll
        for (int i = 0; i < IT; ++i) {
            const uint4 kv = *reinterpret_cast<const uint4*>(sK + swz(i * TPI + tsub, c));
            part[i] = dot8(kv, q2);
        }
        // Reduce-scatter over the CH lanes of a row: afterwards lane c holds
        // token (c >> 1) * TPI + tsub, summed over all chunks.
#pragma unroll
        for (int lv = 0; lv < LOG_IT; ++lv) {
            const int n = IT >> lv;
            const int mask = CH >> (lv + 1);
            const bool hi = (c & mask) != 0;
#pragma unroll
            for (int k = 0; k < n / 2; ++k) {
                const float send = hi ? part[k] : part[k + n / 2];
                const float keep = hi ? part[k + n / 2] : part[k];
                part[k] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
            }
        }
        float sc = part[0] + __shfl_xor_sync(0xffffffffu, part[0], 1);
        const int tok = (c >> 1) * TPI + tsub;
        sc = (tok < valid) ? sc * scale_log2 : -INFINITY;
        // The reference m moves only when a score exceeds it by more than 8
        // (log2 units; see GqaCompute::page), so most pages skip the max
        // reduction and the rescale.
        if (__any_sync(0xffffffffu, sc > m + 8.f)) {
            float pm = sc;
#pragma unroll
            for (int mask = 2; mask < 32; mask <<= 1) pm = fmaxf(pm, __shfl_xor_sync(0xffffffffu, pm, mask));
            const float mn = fmaxf(m, pm);
            const float alpha = ex2(m - mn);
            l *= alpha;
            m = mn;
            const uint64_t a2 = f2_pack(alpha, alpha);
#pragma unroll
            for (int k = 0; k < 4; ++k) o2[k] = f2_fma(o2[k], a2, 0ull);
        }
        const float pe = ex2(sc - m);
        l += (c & 1) ? 0.f : pe;
#pragma unroll
        for (int i = 0; i < IT; ++i) {
            const float pt = __shfl_sync(0xffffffffu, pe, tsub * CH + 2 * i);
            const int t = i * TPI + tsub;
            if (t < valid) {   // rows past the end may hold anything
                const uint4 vv = *reinterpret_cast<const uint4*>(sV + swz(t, c));
                axpy8(o2, f2_pack(pt, pt), vv);
            }
        }
    }

    // Writes the output (a row of one item) or the item's partial (a split
    // row; the merge pass combines them).
    __device__ __forceinline__ void finish(const DecodeParams& p, const PlanEntry& en, int g, int lane)
    {
        float o[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) f2_unpack(o2[k], o[2 * k], o[2 * k + 1]);
#pragma unroll
        for (int mask = CH; mask < 32; mask <<= 1)
#pragma unroll
            for (int k = 0; k < 8; ++k) o[k] += __shfl_xor_sync(0xffffffffu, o[k], mask);
#pragma unroll
        for (int mask = 1; mask < 32; mask <<= 1) l += __shfl_xor_sync(0xffffffffu, l, mask);
        if (en.n_chunks == 1) {
            if (tsub == 0) {
                const float inv = 1.f / l;
                uint4 v;
                v.x = pack_bf16(o[0] * inv, o[1] * inv);
                v.y = pack_bf16(o[2] * inv, o[3] * inv);
                v.z = pack_bf16(o[4] * inv, o[5] * inv);
                v.w = pack_bf16(o[6] * inv, o[7] * inv);
                *reinterpret_cast<uint4*>(p.out + ((int64_t)en.b * p.H_q + g) * D + c * 8) = v;
            }
        } else {
            const int64_t slot = (int64_t)(en.slot_base + en.chunk) * p.H_kv + g;
            if (tsub == 0) {
                float4* dst = reinterpret_cast<float4*>(p.part_o + slot * D + c * 8);
                dst[0] = make_float4(o[0], o[1], o[2], o[3]);
                dst[1] = make_float4(o[4], o[5], o[6], o[7]);
            }
            if (lane == 0) p.part_ml[slot] = make_float2(m, l);
        }
    }
};

// ------------------------------------------------------------ GQA, bf16 MMA
// S^T[16 tokens][8 heads] = K . q^T and O^T[D][8 heads] += V^T . P^T with
// mma.m16n8k16; accumulator columns of a lane are heads 2*(lane&3) and +1.
template <int D>
struct GqaCompute {
    static constexpr int KS = D / 16;
    int G;
    uint32_t qb[KS][2];
    float m0, m1, l0, l1;
    float oacc[KS][4];

    __device__ __forceinline__ void start(const DecodeParams& p, const PlanEntry& en, int g, int lane)
    {
        G = p.G;
        const int n = lane >> 2;
        const uint16_t* qrow = p.q + ((int64_t)en.b * p.H_q + g * G + (n < G ? n : 0)) * D;
#pragma unroll
        for (int ks = 0; ks < KS; ++ks) {
            const uint32_t x0 = *reinterpret_cast<const uint32_t*>(qrow + ks * 16 + 2 * (lane & 3));
            const uint32_t x1 = *reinterpret_cast<const uint32_t*>(qrow + ks * 16 + 8 + 2 * (lane & 3));
            qb[ks][0] = (n < G) ? x0 : 0u;
            qb[ks][1] = (n < G) ? x1 : 0u;
        }
        m0 = m1 = -INFINITY;
        l0 = l1 = 0.f;
#pragma unroll
        for (int mt = 0; mt < KS; ++mt)
#pragma unroll
            for (int k = 0; k < 4; ++k) oacc[mt][k] = 0.f;
    }

    __device__ __forceinline__ void page(uint8_t*, uint8_t*, uint32_t sK, uint32_t sV, int valid,
                                         float scale_log2, int lane)
    {
        // S^T over the D/16 k-steps in four independent accumulator chains
        // (a shorter dependent MMA sequence), summed at the end.
        float sc[4] = {0.f, 0.f, 0.f, 0.f};
        {
            constexpr int NA = KS < 4 ? KS : 4;
            float acc[NA][4];
#pragma unroll
            for (int a = 0; a < NA; ++a)
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[a][k] = 0.f;
            const int r = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                uint32_t a0, a1, a2, a3;
                ldsm_x4(sK + swz(r, ks * 2 + (lane >> 4)), a0, a1, a2, a3);
                mma_bf16_16816(acc[ks % NA], a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
            }
#pragma unroll
            for (int a = 0; a < NA; ++a)
#pragma unroll
                for (int k = 0; k < 4; ++k) sc[k] += acc[a][k];
        }
        // V^T's fragments now, so their shared-memory latency overlaps the
        // softmax.  Rows past the end may hold anything (a NaN pattern would
        // survive a zero weight), so a partial page zeroes their bf16 halves
        // in registers: lane t holds tokens 2(t%4), 2(t%4)+1 in a0/a1 and
        // those + 8 in a2/a3.
        uint32_t vf[KS][4];
        {
            const int r = (lane & 7) + (lane >> 4) * 8;
#pragma unroll
            for (int mt = 0; mt < KS; ++mt)
                ldsm_x4_trans(sV + swz(r, mt * 2 + ((lane >> 3) & 1)), vf[mt][0], vf[mt][1], vf[mt][2], vf[mt][3]);
            if (valid < kPageSize) {
                const int tk = 2 * (lane & 3);
                const uint32_t ma = (tk < valid ? 0x0000ffffu : 0u) | (tk + 1 < valid ? 0xffff0000u : 0u);
                const uint32_t mb = (tk + 8 < valid ? 0x0000ffffu : 0u) | (tk + 9 < valid ? 0xffff0000u : 0u);
#pragma unroll
                for (int mt = 0; mt < KS; ++mt) {
                    vf[mt][0] &= ma;
                    vf[mt][1] &= ma;
                    vf[mt][2] &= mb;
                    vf[mt][3] &= mb;
                }
            }
        }
        const int t0 = lane >> 2, t1 = t0 + 8;
        const bool v0 = t0 < valid, v1 = t1 < valid;
        sc[0] = v0 ? sc[0] * scale_log2 : -INFINITY;
        sc[1] = v0 ? sc[1] * scale_log2 : -INFINITY;
        sc[2] = v1 ? sc[2] * scale_log2 : -INFINITY;
        sc[3] = v1 ? sc[3] * scale_log2 : -INFINITY;
        // The reference m of a head moves only when one of its scores exceeds
        // it by more than 8 (log2 units): the weights 2^(s - m) then stay at
        // most 2^8, far inside the fp32 and bf16 range, and most pages skip
        // the max reduction and the rescale of o and l.  Any reference gives
        // the same o / l; the merge pass takes (o, m, l) with m as that
        // reference.
        float pm0 = fmaxf(sc[0], sc[2]), pm1 = fmaxf(sc[1], sc[3]);
        if (__any_sync(0xffffffffu, pm0 > m0 + 8.f || pm1 > m1 + 8.f)) {
#pragma unroll
            for (int mask = 4; mask < 32; mask <<= 1) {
                pm0 = fmaxf(pm0, __shfl_xor_sync(0xffffffffu, pm0, mask));
                pm1 = fmaxf(pm1, __shfl_xor_sync(0xffffffffu, pm1, mask));
            }
            const float mn0 = fmaxf(m0, pm0), mn1 = fmaxf(m1, pm1);
            const float al0 = ex2(m0 - mn0), al1 = ex2(m1 - mn1);
            l0 *= al0;
            l1 *= al1;
            m0 = mn0;
            m1 = mn1;
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                oacc[mt][0] *= al0;
                oacc[mt][1] *= al1;
                oacc[mt][2] *= al0;
                oacc[mt][3] *= al1;
            }
        }
        const float p0 = ex2(sc[0] - m0), p1 = ex2(sc[1] - m1);
        const float p2 = ex2(sc[2] - m0), p3 = ex2(sc[3] - m1);
        l0 += p0 + p2;
        l1 += p1 + p3;
        // P^T as the B operand: lane needs P[t=2(lane&3)+{0,1}][h=lane>>2] and
        // the same for t+8.  The packed accumulator pairs (tokens 0-7, then
        // 8-15) are 8x8 bf16 tiles [token][head] in the m8n8 fragment layout;
        // their transposes are the B fragments.
        const uint32_t pb0 = movmatrix_trans(pack_bf16(p0, p1));
        const uint32_t pb1 = movmatrix_trans(pack_bf16(p2, p3));
#pragma unroll
        for (int mt = 0; mt < KS; ++mt)
            mma_bf16_16816(oacc[mt], vf[mt][0], vf[mt][1], vf[mt][2], vf[mt][3], pb0, pb1);
    }

    __device__ __forceinline__ void finish(const DecodeParams& p, const PlanEntry& en, int g, int lane)
    {
#pragma unroll
        for (int mask = 4; mask < 32; mask <<= 1) {
            l0 += __shfl_xor_sync(0xffffffffu, l0, mask);
            l1 += __shfl_xor_sync(0xffffffffu, l1, mask);
        }
        const int h0 = 2 * (lane & 3), h1 = h0 + 1;
        const int dlo = lane >> 2;
        if (en.n_chunks == 1) {
            const float i0 = 1.f / l0, i1 = 1.f / l1;
            uint16_t* ob = p.out + ((int64_t)en.b * p.H_q + g * G) * D;
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                const int d0 = mt * 16 + dlo;
                if (h0 < G) {
                    ob[h0 * D + d0] = (uint16_t)(pack_bf16(oacc[mt][0] * i0, 0.f) & 0xffffu);
                    ob[h0 * D + d0 + 8] = (uint16_t)(pack_bf16(oacc[mt][2] * i0, 0.f) & 0xffffu);
                }
                if (h1 < G) {
                    ob[h1 * D + d0] = (uint16_t)(pack_bf16(oacc[mt][1] * i1, 0.f) & 0xffffu);
                    ob[h1 * D + d0 + 8] = (uint16_t)(pack_bf16(oacc[mt][3] * i1, 0.f) & 0xffffu);
                }
            }
        } else {
            const int64_t slot = (int64_t)(en.slot_base + en.chunk) * p.H_kv + g;
            float* po = p.part_o + slot * G * D;
#pragma unroll
            for (int mt = 0; mt < KS; ++mt) {
                const int d0 = mt * 16 + dlo;
                if (h0 < G) {
                    po[h0 * D + d0] = oacc[mt][0];
                    po[h0 * D + d0 + 8] = oacc[mt][2];
                }
                if (h1 < G) {
                    po[h1 * D + d0] = oacc[mt][1];
                    po[h1 * D + d0 + 8] = oacc[mt][3];
                }
            }
            if (lane < 4) {
                if (h0 < G) p.part_ml[slot * G + h0] = make_float2(m0, l0);
                if (h1 < G) p.part_ml[slot * G + h1] = make_float2(m1, l1);
            }
        }
    }
};

// The new token of row (en.b, g), 16 bytes per lane: lanes 0..CH-1 hold K,
// CH..2CH-1 hold V.  Loaded when the row's last item starts, so the load is
// back long before its last page (where waiting for it cost ~2 us under a
// saturated HBM).
template <int D>
__device__ __forceinline__ uint4 load_new_token(const DecodeParams& p, const PlanEntry& en, int g, int lane)
{
    constexpr int CH = D / 8;
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (lane < 2 * CH) {
        const bool is_k = lane < CH;
        const int c = is_k ? lane : lane - CH;
        const int64_t src = ((int64_t)en.b * p.H_kv + g) * D + c * 8;
        v = *reinterpret_cast<const uint4*>((is_k ? p.k_new : p.v_new) + src);
    }
    return v;
}

// The new token (load_new_token's v) into row r of the staged K and V tiles
// and, unless its page id is out of range (already recorded), into the pool
// (fused append).
template <int D>
__device__ __forceinline__ void put_new_token(const DecodeParams& p, const PlanEntry& en, int g, int32_t pid,
                                              const uint4& v, uint8_t* sK, uint8_t* sV, int lane)
{
    constexpr int CH = D / 8;
    const int r = (en.len - 1) % kPageSize;
    if (lane < 2 * CH) {
        const bool is_k = lane < CH;
        const int c = is_k ? lane : lane - CH;
        *reinterpret_cast<uint4*>((is_k ? sK : sV) + swz(r, c)) = v;
        if (pid >= 0 && pid < p.num_pages) {
            const int64_t dst = (((int64_t)pid * p.H_kv + g) * kPageSize + r) * D + c * 8;
            *reinterpret_cast<uint4*>((is_k ? p.pool_k : p.pool_v) + dst) = v;
        }
    }
    __syncwarp();
}

template <int D, bool GQA, bool FUSED>
__global__ void __launch_bounds__(kWarps * 32)
    decode_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                  const DecodeParams p)
{
    using Gm = Geo<D, GQA>;
    constexpr int R = Gm::kRing;
    constexpr int STAGE = Gm::kStageBytes;
    constexpr int TILE = Gm::kTileBytes;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                               ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* ring = smem + warp * R * STAGE;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + Gm::kRingBytes) + warp * R;
    const uint32_t ring_s = smem_addr(ring);

    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < R; ++s) mbar_init(smem_addr(&bars[s]), 1);
        fence_mbar_init();
    }
    if (threadIdx.x == 0) {
        prefetch_tensormap(&tmk);
        prefetch_tensormap(&tmv);
    }
    __syncthreads();
    const uint64_t policy = l2_policy_evict_first();

    uint32_t phase = 0;    // bit s: parity of the next completion of stage s
    uint32_t pending = 0;  // bit s: stage s has a load in flight that was not waited on
    bool ok = true;

    using Comp = typename std::conditional<GQA, GqaCompute<D>, MhaCompute<D>>::type;
    Comp comp;
    // Fused launches depend programmatically on the previous kernel: until
    // griddep_wait() only the plan, page table and cache pages (none of which
    // that kernel writes) are read; q, k_new, v_new and every write come after.
    bool waited = !FUSED;
    bool first_item = true;

    // The first item of every warp is its global warp index; later ones come
    // from the work counter, offset by the number of warps.
    const int n_warps = (int)gridDim.x * kWarps;
    int item = (int)blockIdx.x * kWarps + warp;

    const int n_items = p.n_entries_dev ? min(p.n_items, *p.n_entries_dev * p.H_kv) : p.n_items;
    while (item < n_items) {
        const int e = item / p.H_kv;
        const int g = item - e * p.H_kv;
        // The entry's page ids sit at a fixed stride, so they load alongside
        // the entry.  Windows of 32: lane i holds page w*32 + i of the current
        // window; the next window is fetched 24 pages ahead.
        const int32_t* pt_row = p.item_pages + (int64_t)e * p.page_stride;
        auto load_window = [&](int w0) { return (w0 + lane < p.page_stride) ? pt_row[w0 + lane] : 0; };
        int32_t pid_cur = load_window(0);
        int32_t pid_next = 0;
        const PlanEntry en = p.plan[e];
        const int np = en.n_pages;

        auto issue = [&](int j, int s) {
            if ((j & 31) == 8 && j + 24 < np) pid_next = load_window(j + 24);
            if ((j & 31) == 0 && j > 0) pid_cur = pid_next;
            int32_t pid = __shfl_sync(0xffffffffu, pid_cur, j & 31);
            if (pid < 0 || pid >= p.num_pages) {
                if (lane == 0) atomicOr(p.err, 1);
                pid = 0;
            }
            if (lane == 0) {
                const uint32_t bar = smem_addr(&bars[s]);
                const uint32_t dst = ring_s + s * STAGE;
                const int32_t y = (pid * p.H_kv + g) * kPageSize;
                mbar_arrive_expect_tx(bar, STAGE);
                if (p.kv_map) {
                    tma_load_4d(dst, &tmk, 0, y, 0, 0, bar, policy);
                } else {
                    tma_load_3d(dst, &tmk, 0, y, 0, bar, policy);
                    tma_load_3d(dst + TILE, &tmv, 0, y, 0, bar, policy);
                }
            }
        };

        const int pre = np < R ? np : R;
        __syncwarp();
        for (int j = 0; j < pre; ++j) issue(j, j);
        pending = (1u << pre) - 1u;
        int ramp0 = R;   // first page of the L2 ramp at the wait's return
        if (!waited && p.prev_tag && np > R && p.kv_map) {
            unsigned smid;
            asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
            const uint32_t want = *p.step_no * 65536u + p.prev_tag;
            const volatile uint32_t* flag = p.start_flags + (smid % (unsigned)p.num_sms) * 32;
            const uint64_t t0 = global_timer_ns();
            bool seen = false;
            while (true) {
                seen = *flag == want;
                if (seen || global_timer_ns() - t0 > kEarlyPollLimitNs) break;
                __nanosleep(128);
            }
            if (seen) {
                for (int j = R; j < np && j < R + kEarlyL2Pages; ++j) {
                    int32_t pid = __shfl_sync(0xffffffffu, pid_cur, j & 31);
                    if (pid < 0 || pid >= p.num_pages) pid = 0;   // recorded when its load is issued
                    if (lane == 0) tma_prefetch_l2_4d(&tmk, 0, (pid * p.H_kv + g) * kPageSize, 0, 0);
                }
                ramp0 = R + kEarlyL2Pages;
            }
        }
        if (!waited) {
            griddep_wait();
            griddep_launch_dependents();
            waited = true;
        }
        if (first_item && p.kv_map) {
            // The ring holds this item's first R pages (loaded before the
            // wait when chained); the next ones go into L2 now.
            for (int j = ramp0; j < np && j < ramp0 + kRampL2Pages; ++j) {
                int32_t pid = __shfl_sync(0xffffffffu, pid_cur, j & 31);
                if (pid < 0 || pid >= p.num_pages) pid = 0;   // recorded when its load is issued
                if (lane == 0) tma_prefetch_l2_4d(&tmk, 0, (pid * p.H_kv + g) * kPageSize, 0, 0);
            }
        }
        first_item = false;
        comp.start(p, en, g, lane);
        const bool last_chunk = en.chunk == en.n_chunks - 1;
        uint4 new_kv = make_uint4(0u, 0u, 0u, 0u);
        if constexpr (FUSED)
            if (last_chunk) new_kv = load_new_token<D>(p, en, g, lane);

        for (int j = 0; j < np; ++j) {
            const int s = j % R;
            const bool w = mbar_wait_bounded(smem_addr(&bars[s]), (phase >> s) & 1u, kWaitLimitNs);
            if (!__all_sync(0xffffffffu, w)) {
                ok = false;
                break;
            }
            phase ^= 1u << s;
            pending &= ~(1u << s);
            const int valid = min(kPageSize, en.len - (en.first_page + j) * kPageSize);
            uint8_t* sK = ring + s * STAGE;
            // Generic-proxy writes into the stage (the new token's row) must be
            // ordered before the next TMA write to it; plain reads need no
            // fence (their values are consumed first).
            bool wrote = false;
            if constexpr (FUSED) {
                // the issue side has not moved past this page's id window
                if (last_chunk && j == np - 1) {
                    int32_t pid = __shfl_sync(0xffffffffu, pid_cur, j & 31);
                    put_new_token<D>(p, en, g, pid, new_kv, sK, sK + TILE, lane);
                    wrote = true;
                }
            }
            comp.page(sK, sK + TILE, ring_s + s * STAGE, ring_s + s * STAGE + TILE, valid, p.scale_log2, lane);
            if (wrote) fence_proxy_async_smem();
            __syncwarp();
            if (j + R < np) {
                issue(j + R, s);
                pending |= 1u << s;
            }
        }
        if (!ok) break;
        comp.finish(p, en, g, lane);
        if (lane == 0) item = n_warps + (int)atomicAdd(&p.queue[0], 1u);
        item = __shfl_sync(0xffffffffu, item, 0);
    }

    if (!ok && lane == 0) atomicOr(p.err, 2);
    // Let every load this warp issued land before the warp leaves.
#pragma unroll
    for (int s = 0; s < R; ++s)
        if (pending & (1u << s)) mbar_wait_bounded(smem_addr(&bars[s]), (phase >> s) & 1u, kWaitLimitNs);
    __syncwarp();

    // Every warp completes only after the launch it depends on has (so a
    // launch's completion always implies its predecessor's).  Then one thread
    // resets the work counter of the next launch: the previous launch used it
    // and has completed.  The next launch fetches from it only after its own
    // dependency wait, i.e. after this launch has completed.
    if (!waited) griddep_wait();
    if (blockIdx.x == 0 && threadIdx.x == 0 && p.queue_next) *p.queue_next = 0u;
}

}  // namespace

}  // namespace kvd
