// Forward GEMMs: Z/H = sigma-epilogue of X A^T (EPI_ZH) and Y = H B^T (EPI_STORE);
// both operands K-major.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {
template cudaError_t launch_gemm<128, 1, false, false, EPI_ZH>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_ZH>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_ZH>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, false, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
}  // namespace cola
