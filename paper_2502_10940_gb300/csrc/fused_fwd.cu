// The single-kernel forward of a CoLA layer with r <= 128 (fused_fwd.cuh):
// its launcher, instantiated for r = 64 and r = 128.
#include <cuda_runtime.h>

#include <atomic>

#include "fused_fwd.cuh"

namespace cola {

template <int R>
static cudaError_t launch_fused_fwd_r(const FusedFwdParams& p, int grid, bool pdl, cudaStream_t stream)
{
    constexpr int smem = FusedCfg<R>::SMEM_BYTES;
    auto kern = fused_fwd_kernel<R>;
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

cudaError_t launch_fused_fwd(const FusedFwdParams& p, int r, int grid, bool pdl, cudaStream_t stream)
{
    if (r == 64) return launch_fused_fwd_r<64>(p, grid, pdl, stream);
    if (r == 128) return launch_fused_fwd_r<128>(p, grid, pdl, stream);
    return cudaErrorInvalidValue;
}

}  // namespace cola
