// Forward GEMMs: Z/H = sigma-epilogue of X A^T (EPI_ZH) and Y = H B^T (EPI_STORE);
// both operands K-major.  Also the elementwise H = sigma(Z) that the CoLA-M
// up-projection recompute runs before its Y GEMM.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {
template cudaError_t launch_gemm<128, 1, false, false, EPI_ZH, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, false, EPI_ZH, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, false, EPI_ZH, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_ZH, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_ZH, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_ZH, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, true, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, true, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH, true, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_STORE, true>(const GemmBatch&, int, bool, cudaStream_t);

// sigma of 8 bf16 values (one 16-byte vector), with the logistic's form L
template <int S, int L>
__device__ __forceinline__ uint4 sigma8(const uint4 z)
{
    uint4 h;
    h.x = pack_bf16x2(act_sigma<S, L>(bf16_lo(z.x)), act_sigma<S, L>(bf16_hi(z.x)));
    h.y = pack_bf16x2(act_sigma<S, L>(bf16_lo(z.y)), act_sigma<S, L>(bf16_hi(z.y)));
    h.z = pack_bf16x2(act_sigma<S, L>(bf16_lo(z.z)), act_sigma<S, L>(bf16_hi(z.z)));
    h.w = pack_bf16x2(act_sigma<S, L>(bf16_lo(z.w)), act_sigma<S, L>(bf16_hi(z.w)));
    return h;
}

// H = bf16(sigma(Z)) over `vecs` groups of 8 bf16, each a 16-byte vector;
// sigma is evaluated exactly as in the Z/H epilogue (same function on the
// same bf16 inputs), so the result is bit-identical to the forward's H.
template <int S>
__global__ void __launch_bounds__(256) sigma_kernel(const uint4* __restrict__ Z, uint4* __restrict__ H, long long vecs)
{
    grid_dependency_wait();            // Z may come from the kernel launched just before
    grid_launch_dependents();
    const long long stride = static_cast<long long>(gridDim.x) * blockDim.x;
    for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < vecs; i += stride) {
        const uint4 z = __ldg(Z + i);
        const uint32_t zw[4] = {z.x, z.y, z.z, z.w};
        // the logistic's tanh form alone where no input lies below its floor
        H[i] = (S == SIG_SILU && !below_tanh_floor(zw)) ? sigma8<S, LOGI_TANH>(z) : sigma8<S, LOGI_SELECT>(z);
    }
}

cudaError_t launch_sigma(const void* Z, void* H, long long elems, int sigma, int sms, cudaStream_t stream)
{
    const long long vecs = elems / 8;
    long long blocks = (vecs + 255) / 256;
    if (blocks > 8LL * sms) blocks = 8LL * sms;   // grid-stride beyond 8 blocks per SM
    if (blocks < 1) blocks = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const uint4* z = static_cast<const uint4*>(Z);
    uint4* h = static_cast<uint4*>(H);
    if (sigma == SIG_SILU) return cudaLaunchKernelEx(&cfg, sigma_kernel<SIG_SILU>, z, h, vecs);
    if (sigma == SIG_GELU) return cudaLaunchKernelEx(&cfg, sigma_kernel<SIG_GELU>, z, h, vecs);
    return cudaLaunchKernelEx(&cfg, sigma_kernel<SIG_IDENTITY>, z, h, vecs);
}
}  // namespace cola
