// gemm_launch.cuh -- host-side launcher of the GEMM kernel template.  The
// kernel translation units (gemm_*.cu) instantiate it explicitly; the ABI
// translation unit only sees the declarations.
#pragma once
#include <cuda_runtime.h>

#include "gemm.cuh"

namespace cola {

// map_d / map_d2: bf16 output boxes {32, 32} (64-byte swizzle); map_z: the
// saved Z that EPI_DSIGMA reads, same box geometry.  Maps an epilogue does
// not use may be any valid map.
// pdl: launch with programmatic stream serialization (the prologue overlaps
// the previous kernel's tail).  Worth it for short launches only.
template <int BN, int MSUB, bool A_MN, bool B_MN, int EPI>
cudaError_t launch_gemm(const CUtensorMap& map_a, const CUtensorMap& map_b, const CUtensorMap& map_d,
                        const CUtensorMap& map_d2, const CUtensorMap& map_z, const GemmParams& p, int grid,
                        bool pdl, cudaStream_t stream);

cudaError_t launch_splitk_reduce(const float* part, int splits, long long part_stride, int ldp, int M, int N,
                                 void* out, long long ldo, int accumulate_f32, int grid, cudaStream_t stream);

#ifdef COLA_DEFINE_LAUNCHERS
template <int BN, int MSUB, bool A_MN, bool B_MN, int EPI>
cudaError_t launch_gemm(const CUtensorMap& map_a, const CUtensorMap& map_b, const CUtensorMap& map_d,
                        const CUtensorMap& map_d2, const CUtensorMap& map_z, const GemmParams& p, int grid,
                        bool pdl, cudaStream_t stream)
{
    constexpr int smem = GemmCfg<BN, MSUB>::SMEM_BYTES;
    auto kern = gemm_kernel<BN, MSUB, A_MN, B_MN, EPI>;
    // the opt-in shared-memory size is a per-device function attribute
    static unsigned long long configured = 0;   // bit d: set on device d
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 64 || !((configured >> dev) & 1ull)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        if (dev < 64) configured |= 1ull << dev;
    }
    // programmatic stream serialization: this kernel's prologue may overlap
    // the tail of the previous kernel in the stream (see grid_dependency_wait)
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
    return cudaLaunchKernelEx(&cfg, kern, map_a, map_b, map_d, map_d2, map_z, p);
}
#endif

}  // namespace cola
