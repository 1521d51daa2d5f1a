// gemm_launch.cuh -- host-side launcher of the GEMM kernel template.  The
// kernel translation units (gemm_*.cu) instantiate it explicitly; the ABI
// translation unit only sees the declarations.
#pragma once
#include <cuda_runtime.h>

#include <atomic>

#include "gemm.cuh"

namespace cola {

// Launch the GEMM kernel over a batch of problems (see GemmBatch).  pdl:
// launch with programmatic stream serialization (the prologue overlaps the
// previous kernel's tail).  PAIR: clusters of two CTAs (grid even), each
// pair running one 256-row tile with tcgen05 cta_group::2.
// SIG: the activation the epilogue applies (EPI_ZH, EPI_DSIGMA, EPI_DSIGMA_H
// are compiled once per activation; the other kinds take SIG_IDENTITY).
template <int BN, int MSUB, bool A_MN, bool B_MN, int EPI, bool PAIR = false, int SIG = SIG_IDENTITY>
cudaError_t launch_gemm(const GemmBatch& batch, int grid, bool pdl, cudaStream_t stream);

// One fixed-order reduction of fp32 split partials into a result: a weight
// gradient, a split-K output GEMM (bf16), or the split-K Z/H GEMM (zh: Z =
// bf16(sum) into `out` when not null, H = bf16(sigma(Z)) into `out2`).
struct ReduceJob {
    const float* part;          // splits slabs of part_stride elements
    long long part_stride;
    int ldp;                    // row pitch of a slab
    int M, N;
    void* out;                  // bf16 (or fp32 when accumulating)
    void* out2;                 // zh: H
    long long ldo;              // row pitch of out and out2
    long long group_begin;      // first 4-column group of this job in the launch (set by the launcher)
};

struct ReduceBatch {
    ReduceJob job[MAX_GROUP];
    int count;
    int splits;
    int accumulate_f32;
    int zh;                     // 1: the Z/H epilogue (out = Z or null, out2 = H)
    int sigma;                  // zh: the activation
    long long groups;           // 4-column groups of all jobs (set by the launcher)
};

cudaError_t launch_splitk_reduce(ReduceBatch& batch, cudaStream_t stream);

// The tail reduce of an EPI_TAIL launch: each split tail tile is the sum of
// its pieces' partial slots, added in piece order (so the result is
// deterministic), stored as bf16 into its problem's output.
constexpr int MAX_TAIL_TILES = 160;   // tail tiles are fewer than the CTA slots (<= 151 on GB300)

struct TailTile {
    int g;          // problem
    int m0, n0;     // first row and column of the tile in the problem's output
    int lo_slot;    // partial slot of its first piece; the others follow it
    int count;      // pieces
};

struct TailReduce {
    const float* part;              // partial slots of tile_rows x tile_cols fp32 each
    int tile_rows, tile_cols;
    void* out[MAX_GROUP];           // bf16 outputs of the launch's problems
    long long ldo[MAX_GROUP];
    int M[MAX_GROUP], N[MAX_GROUP];
    int ntiles;
    TailTile tile[MAX_TAIL_TILES];
};

cudaError_t launch_tail_reduce(const TailReduce& r, int sms, cudaStream_t stream);

// H = bf16(sigma(Z)) elementwise over `elems` bf16 values (a multiple of 8;
// both pointers 16-byte aligned).
cudaError_t launch_sigma(const void* Z, void* H, long long elems, int sigma, int sms, cudaStream_t stream);

#ifdef COLA_DEFINE_LAUNCHERS
template <int BN, int MSUB, bool A_MN, bool B_MN, int EPI, bool PAIR, int SIG>
cudaError_t launch_gemm(const GemmBatch& batch, int grid, bool pdl, cudaStream_t stream)
{
    constexpr int smem = GemmCfg<BN, MSUB, PAIR>::SMEM_BYTES;
    auto kern = gemm_kernel<BN, MSUB, A_MN, B_MN, EPI, PAIR, SIG>;
    // the opt-in shared-memory size is a per-device function attribute; host
    // threads may launch concurrently, so the set of configured devices is atomic
    static std::atomic<unsigned long long> configured{0};   // bit d: set on device d
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
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (PAIR) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = 2;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    return cudaLaunchKernelEx(&cfg, kern, batch);
}
#endif

}  // namespace cola
