// Weight-gradient GEMMs dB = dY^T H and dA = dZ^T X: the reduction runs over
// the n tokens, both operands are token-major activations read MN-major, and
// the token range is split across CTAs into fp32 partial slabs that
// splitk_reduce_kernel sums in a fixed order.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {

// ------------------------------------------------ split-K reduction
// out[i, j] = sum over s = 0..splits-1 (in that order) of part[s][i][j];
// bf16 store, or fp32 accumulate (out += sum) when accumulate_f32.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, int splits, long long part_stride,
                                     int ldp, int M, int N, void* out, long long ldo, int accumulate_f32)
{
    const int groups = (N + 3) / 4;
    const long long total = static_cast<long long>(M) * groups;
    for (long long g = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; g < total;
         g += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int i = static_cast<int>(g / groups);
        const int j = static_cast<int>(g - static_cast<long long>(i) * groups) * 4;
        const float* src = part + static_cast<long long>(i) * ldp + j;
        float4 acc = *reinterpret_cast<const float4*>(src);
        for (int s = 1; s < splits; ++s) {
            const float4 t = *reinterpret_cast<const float4*>(src + s * part_stride);
            acc.x += t.x;
            acc.y += t.y;
            acc.z += t.z;
            acc.w += t.w;
        }
        const float a[4] = {acc.x, acc.y, acc.z, acc.w};
        const int valid = min(4, N - j);
        if (accumulate_f32) {
            float* o = reinterpret_cast<float*>(out) + static_cast<long long>(i) * ldo + j;
            for (int e = 0; e < valid; ++e) o[e] += a[e];
        } else {
            __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(out) + static_cast<long long>(i) * ldo + j;
            if (valid == 4 && ((reinterpret_cast<uintptr_t>(o) & 7) == 0)) {
                uint2 pk = make_uint2(pack_bf16x2(a[0], a[1]), pack_bf16x2(a[2], a[3]));
                *reinterpret_cast<uint2*>(o) = pk;
            } else {
                for (int e = 0; e < valid; ++e) o[e] = __float2bfloat16_rn(a[e]);
            }
        }
    }
}


template cudaError_t launch_gemm<128, true, true, EPI_F32>(const CUtensorMap&, const CUtensorMap&, const CUtensorMap&,
                                                           const CUtensorMap&, const GemmParams&, int,
                                                            cudaStream_t);
template cudaError_t launch_gemm<256, true, true, EPI_F32>(const CUtensorMap&, const CUtensorMap&, const CUtensorMap&,
                                                           const CUtensorMap&, const GemmParams&, int,
                                                            cudaStream_t);

cudaError_t launch_splitk_reduce(const float* part, int splits, long long part_stride, int ldp, int M, int N,
                                 void* out, long long ldo, int accumulate_f32, int grid, cudaStream_t stream)
{
    splitk_reduce_kernel<<<grid, 256, 0, stream>>>(part, splits, part_stride, ldp, M, N, out, ldo, accumulate_f32);
    return cudaGetLastError();
}
}  // namespace cola
