// Weight-gradient GEMMs dB = dY^T H and dA = dZ^T X: the reduction runs over
// the n tokens, both operands are token-major activations read MN-major, and
// the token range is split across CTAs into fp32 partial slabs that
// splitk_reduce_kernel sums in a fixed order (or, unsplit, the epilogue
// stores the bf16 gradient directly).
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {

// ------------------------------------------------ split-K reduction
// out[i, j] = sum over s = 0..splits-1 of part[s][i][j], bf16 store or fp32
// accumulate (out += sum), for up to MAX_GROUP gradients in one launch.  One
// block covers 32 groups of 4 consecutive columns of one gradient; its
// `ways` = min(8, splits) warps take the splits s = w, w + ways, ... (one warp
// reads 512 contiguous bytes of a slab per split), and the per-warp sums of a
// group are added in the fixed order w = 0..ways-1.  Every run adds the same
// numbers in the same order: the result is deterministic.
constexpr int RED_GROUPS = 32;
constexpr int RED_WAYS = 8;

__global__ void __launch_bounds__(RED_GROUPS * RED_WAYS) splitk_reduce_kernel(const __grid_constant__ ReduceBatch rb)
{
    __shared__ float4 red[RED_WAYS][RED_GROUPS];
    grid_dependency_wait();            // the partials come from the GEMM launched just before
    grid_launch_dependents();
    int jb = 0;
#pragma unroll
    for (int j = 1; j < MAX_GROUP; ++j)
        if (j < rb.count && static_cast<long long>(blockIdx.x) >= rb.job[j].block_begin) jb = j;
    const ReduceJob& job = rb.job[jb];
    const int splits = rb.splits;
    const int ways = blockDim.x >> 5;
    const int gl = threadIdx.x & 31;
    const int way = threadIdx.x >> 5;
    const int groups_per_row = (job.N + 3) / 4;
    const long long total = static_cast<long long>(job.M) * groups_per_row;
    const long long g = (static_cast<long long>(blockIdx.x) - job.block_begin) * RED_GROUPS + gl;
    int i = 0, j = 0;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (g < total) {
        i = static_cast<int>(g / groups_per_row);
        j = static_cast<int>(g - static_cast<long long>(i) * groups_per_row) * 4;
        const float* src = job.part + static_cast<long long>(i) * job.ldp + j;
#pragma unroll 4
        for (int sp = way; sp < splits; sp += ways) {
            const float4 t = __ldg(reinterpret_cast<const float4*>(src + sp * job.part_stride));
            acc.x += t.x;
            acc.y += t.y;
            acc.z += t.z;
            acc.w += t.w;
        }
    }
    if (ways > 1) {
        red[way][gl] = acc;
        __syncthreads();
        if (way != 0) return;
        acc = red[0][gl];
        for (int w = 1; w < ways; ++w) {
            const float4 t = red[w][gl];
            acc.x += t.x;
            acc.y += t.y;
            acc.z += t.z;
            acc.w += t.w;
        }
    }
    if (g >= total) return;
    const float v[4] = {acc.x, acc.y, acc.z, acc.w};
    const int valid = min(4, job.N - j);
    if (rb.accumulate_f32) {
        float* o = reinterpret_cast<float*>(job.out) + static_cast<long long>(i) * job.ldo + j;
        for (int e = 0; e < valid; ++e) o[e] += v[e];
    } else {
        __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(job.out) + static_cast<long long>(i) * job.ldo + j;
        if (valid == 4 && ((reinterpret_cast<uintptr_t>(o) & 7) == 0)) {
            *reinterpret_cast<uint2*>(o) = make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
        } else {
            for (int e = 0; e < valid; ++e) o[e] = __float2bfloat16_rn(v[e]);
        }
    }
}

template cudaError_t launch_gemm<128, 1, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_STORE, true>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_F32, true>(const GemmBatch&, int, bool, cudaStream_t);

cudaError_t launch_splitk_reduce(ReduceBatch& rb, cudaStream_t stream)
{
    long long blocks = 0;
    for (int j = 0; j < rb.count; ++j) {
        rb.job[j].block_begin = blocks;
        const long long groups = static_cast<long long>(rb.job[j].M) * ((rb.job[j].N + 3) / 4);
        blocks += (groups + RED_GROUPS - 1) / RED_GROUPS;
    }
    const int ways = rb.splits < RED_WAYS ? rb.splits : RED_WAYS;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(RED_GROUPS * ways);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, splitk_reduce_kernel, rb);
}

}  // namespace cola
