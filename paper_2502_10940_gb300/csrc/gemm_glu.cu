// Gated-MLP GEMMs (Fig. 4: LLaMA's MLP multiplies its gate and up
// projections element-wise; Sec. 3.2 keeps that product when both become
// CoLA layers).  Forward (EPI_GLU): Y_gate = H_gate B_gate^T and
// Y_up = H_up B_up^T of one output tile in two accumulators of one CTA (CTA
// pair), stored as M = Y_gate * Y_up; both operands K-major: 256 x 256 or
// 256 x 128 tiles on CTA pairs, 128 x 128 tiles on single CTAs.  Backward (EPI_GLU_BWD): the down layer's dX GEMM, whose epilogue
// turns dM into dY_gate = dM * Y_up and dY_up = dM * Y_gate; A operand
// K-major, B operand (the down layer's A factor read transposed) MN-major.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {
template cudaError_t launch_gemm<128, 1, false, false, EPI_GLU>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_GLU, true>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, false, EPI_GLU, true>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, false, true, EPI_GLU_BWD>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_GLU_BWD>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, false, true, EPI_GLU_BWD>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, true, EPI_GLU_BWD, true>(const GemmBatch&, int, bool, cudaStream_t);
}  // namespace cola
