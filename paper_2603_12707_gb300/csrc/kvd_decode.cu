// Launch side of the split pass: kernel attributes, occupancy, register
// counts and the (programmatic dependent) launches of decode_kernel
// (kvd_decode_kernel.cuh).
#include <algorithm>

#include "kvd_decode_kernel.cuh"

namespace kvd {

namespace {

template <int D, bool GQA, bool FUSED>
cudaError_t prepare_variant()
{
    static cudaError_t status = cudaFuncSetAttribute(decode_kernel<D, GQA, FUSED>,
                                                     cudaFuncAttributeMaxDynamicSharedMemorySize, Geo<D, GQA>::kSmem);
    return status;
}

template <int D, bool GQA>
cudaError_t variant_info(DecodeVariant* v)
{
    cudaError_t e = prepare_variant<D, GQA, false>();
    if (e == cudaSuccess) e = prepare_variant<D, GQA, true>();
    if (e != cudaSuccess) return e;
    v->warps = kWarps;
    v->smem_bytes = Geo<D, GQA>::kSmem;
    cudaFuncAttributes a0, a1;
    e = cudaFuncGetAttributes(&a0, decode_kernel<D, GQA, false>);
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&a1, decode_kernel<D, GQA, true>);
    if (e != cudaSuccess) return e;
    v->regs = std::max(a0.numRegs, a1.numRegs);
    return cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v->ctas_per_sm, decode_kernel<D, GQA, false>, kWarps * 32,
                                                         Geo<D, GQA>::kSmem);
}

template <int D, bool GQA>
cudaError_t launch_variant(bool fused, bool pdl, int grid, const CUtensorMap& tk, const CUtensorMap& tv,
                           const DecodeParams& p, cudaStream_t st)
{
    if (!fused) {
        cudaError_t e = prepare_variant<D, GQA, false>();
        if (e != cudaSuccess) return e;
        decode_kernel<D, GQA, false><<<grid, kWarps * 32, Geo<D, GQA>::kSmem, st>>>(tk, tv, p);
        return cudaGetLastError();
    }
    cudaError_t e = prepare_variant<D, GQA, true>();
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kWarps * 32);
    cfg.dynamicSmemBytes = Geo<D, GQA>::kSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, decode_kernel<D, GQA, true>, tk, tv, p);
}

}  // namespace

cudaError_t decode_variant_info(int D, bool gqa, DecodeVariant* v)
{
    if (D == 128) return gqa ? variant_info<128, true>(v) : variant_info<128, false>(v);
    if (D == 64) return gqa ? variant_info<64, true>(v) : variant_info<64, false>(v);
    return cudaErrorInvalidValue;
}

cudaError_t launch_decode(int D, bool gqa, bool fused, bool pdl, int grid, const CUtensorMap& tk,
                          const CUtensorMap& tv, const DecodeParams& p, cudaStream_t st)
{
    if (D == 128) return gqa ? launch_variant<128, true>(fused, pdl, grid, tk, tv, p, st)
                             : launch_variant<128, false>(fused, pdl, grid, tk, tv, p, st);
    if (D == 64) return gqa ? launch_variant<64, true>(fused, pdl, grid, tk, tv, p, st)
                            : launch_variant<64, false>(fused, pdl, grid, tk, tv, p, st);
    return cudaErrorInvalidValue;
}

}  // namespace kvd
