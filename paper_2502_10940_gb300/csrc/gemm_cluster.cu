// The cluster-reduced split-K GEMM (splitk_cluster.cuh): its launcher, for
// the weight gradients (token-major, MN-major operands).
#include <cuda_runtime.h>

#include <atomic>

#define COLA_DEFINE_CLUSTER_KERNEL
#include "splitk_cluster.cuh"

namespace cola {

cudaError_t launch_splitk_cluster(const CredBatch& b, bool pdl, cudaStream_t stream)
{
    if (b.S < 1 || b.S > MAX_CLUSTER || b.tiles < 1) return cudaErrorInvalidValue;
    constexpr int smem = CredCfg::SMEM_BYTES;
    auto kern = splitk_cluster_kernel;
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
    cfg.gridDim = dim3(static_cast<unsigned>(b.tiles * b.S));
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = static_cast<unsigned>(b.S);
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, b);
}

}  // namespace cola
