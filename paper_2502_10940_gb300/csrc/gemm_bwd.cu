// Backward activation-gradient GEMMs: dZ = (dY B) * sigma'(Z) (EPI_DSIGMA; with
// H = sigma(Z) for CoLA-M, EPI_DSIGMA_H) and
// dX = dZ A (EPI_STORE); A operand K-major, B operand (a weight read
// transposed) MN-major.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, true, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, true, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA, true, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA_H, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA_H, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_DSIGMA_H, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA_H, false, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA_H, false, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_DSIGMA_H, false, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, true, SIG_IDENTITY>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, true, SIG_SILU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_DSIGMA_H, true, SIG_GELU>(
    const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_STORE, true>(const GemmBatch&, int, bool, cudaStream_t);
}  // namespace cola
