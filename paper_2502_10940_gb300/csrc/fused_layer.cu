// The single-kernel forward and backward passes of a CoLA layer with
// r <= 128 (fused_layer.cuh): their launcher, instantiated for r = 64 and
// r = 128 in both directions and for each activation.
#include <cuda_runtime.h>

#include <atomic>

#include "fused_layer.cuh"

namespace cola {

template <int R, bool BWD, int SIG>
static cudaError_t launch_fused_layer_r(const FusedParams& p, int grid, bool pdl, cudaStream_t stream)
{
    constexpr int smem = FusedCfg<R>::SMEM_BYTES;
    auto kern = fused_layer_kernel<R, BWD, SIG>;
    static std::atomic<unsigned long long> configured{0};   // bit d: attribute set on device d
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 64 || !((configured.load(std::memory_order_acquire) >> dev) & 1ull)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        if (dev < 64) configured.fetch_or(1ull << dev, std::memory_order_acq_rel);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, p);
}

template <int SIG>
static cudaError_t launch_fused_layer_s(const FusedParams& p, int r, bool bwd, int grid, bool pdl,
                                       cudaStream_t stream)
{
    if (r == 64) return bwd ? launch_fused_layer_r<64, true, SIG>(p, grid, pdl, stream)
                            : launch_fused_layer_r<64, false, SIG>(p, grid, pdl, stream);
    if (r == 128) return bwd ? launch_fused_layer_r<128, true, SIG>(p, grid, pdl, stream)
                             : launch_fused_layer_r<128, false, SIG>(p, grid, pdl, stream);
    return cudaErrorInvalidValue;
}

cudaError_t launch_fused_layer(const FusedParams& p, int r, bool bwd, int grid, bool pdl, cudaStream_t stream)
{
    switch (p.sigma) {
    case SIG_SILU: return launch_fused_layer_s<SIG_SILU>(p, r, bwd, grid, pdl, stream);
    case SIG_GELU: return launch_fused_layer_s<SIG_GELU>(p, r, bwd, grid, pdl, stream);
    case SIG_IDENTITY: return launch_fused_layer_s<SIG_IDENTITY>(p, r, bwd, grid, pdl, stream);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace cola
