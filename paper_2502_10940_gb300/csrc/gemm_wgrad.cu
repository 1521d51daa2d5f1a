// Weight-gradient GEMMs dB = dY^T H and dA = dZ^T X: the reduction runs over
// the n tokens, and both operands are token-major activations read MN-major.
// bf16 gradients either run their tiles whole in waves and split only the
// tiles of the last, partial wave over the tokens (EPI_TAIL; tail_reduce_kernel
// sums the pieces), or split every tile's token range uniformly into fp32
// partial slabs that splitk_reduce_kernel sums in a fixed order; fp32
// gradients accumulated into always take the uniform split.  The same
// reduce finishes the split-K forward GEMMs of small launches (instantiated
// here too), applying the Z/H epilogue for the Z GEMM.
#define COLA_DEFINE_LAUNCHERS
#include "gemm_launch.cuh"

namespace cola {

// ------------------------------------------------ split-K reduction
// out[i, j] = sum over s = 0..splits-1 of part[s][i][j], bf16 store or fp32
// accumulate (out += sum), for up to MAX_GROUP gradients in one launch.  The
// groups of 4 consecutive columns of all gradients form one index space that
// a grid of up to 8 CTAs per SM strides through; each thread sums one group's
// splits in the fixed order s = 0, 1, ..., splits-1 (loads issued RED_BATCH at
// a time), so every run adds the same numbers in the same order: the result
// is deterministic.  A batch of 4 keeps the kernel at 40 registers, so that 6
// CTAs fit per SM: more loads are in flight than with batches of 8 at 3 CTAs
// per SM (measured: the 7B down-projection layer's reduce 68 -> 51 us, the 1B
// one 25 -> 18 us, with bit-identical results).
constexpr int RED_THREADS = 256;
constexpr int RED_BATCH = 4;

// ZH: the Z/H epilogue of a split-K Z GEMM with activation SIG (one kernel
// per activation, as the GEMM epilogues); without it the plain sums.
template <bool ZH, int SIG>
__global__ void __launch_bounds__(RED_THREADS) splitk_reduce_kernel(const __grid_constant__ ReduceBatch rb)
{
    grid_dependency_wait();            // the partials come from the GEMM launched just before
    grid_launch_dependents();
    const long long stride = static_cast<long long>(gridDim.x) * RED_THREADS;
    for (long long g = static_cast<long long>(blockIdx.x) * RED_THREADS + threadIdx.x; g < rb.groups; g += stride) {
        int jb = 0;
#pragma unroll
        for (int j = 1; j < MAX_GROUP; ++j)
            if (j < rb.count && g >= rb.job[j].group_begin) jb = j;
        const ReduceJob& job = rb.job[jb];
        const int groups_per_row = (job.N + 3) / 4;
        const long long local = g - job.group_begin;
        const int i = static_cast<int>(local / groups_per_row);
        const int j = static_cast<int>(local - static_cast<long long>(i) * groups_per_row) * 4;
        const float* src = job.part + static_cast<long long>(i) * job.ldp + j;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s0 = 0; s0 < rb.splits; s0 += RED_BATCH) {
            float4 t[RED_BATCH];
#pragma unroll
            for (int b = 0; b < RED_BATCH; ++b)
                if (s0 + b < rb.splits) t[b] = __ldg(reinterpret_cast<const float4*>(src + (s0 + b) * job.part_stride));
#pragma unroll
            for (int b = 0; b < RED_BATCH; ++b) {
                if (s0 + b < rb.splits) {
                    acc.x += t[b].x;
                    acc.y += t[b].y;
                    acc.z += t[b].z;
                    acc.w += t[b].w;
                }
            }
        }
        const float v[4] = {acc.x, acc.y, acc.z, acc.w};
        const int valid = min(4, job.N - j);
        if (ZH) {
            // Z = bf16(sum), H = bf16(sigma(bf16 Z)): the split-K form of the Z/H epilogue
            const uint32_t z01 = pack_bf16x2(v[0], v[1]), z23 = pack_bf16x2(v[2], v[3]);
            const uint32_t h01 = pack_bf16x2(act_sigma<SIG>(bf16_lo(z01)), act_sigma<SIG>(bf16_hi(z01)));
            const uint32_t h23 = pack_bf16x2(act_sigma<SIG>(bf16_lo(z23)), act_sigma<SIG>(bf16_hi(z23)));
            const long long off = static_cast<long long>(i) * job.ldo + j;   // N = count r: 4 | N
            if (job.out) *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(job.out) + off) = make_uint2(z01, z23);
            *reinterpret_cast<uint2*>(reinterpret_cast<__nv_bfloat16*>(job.out2) + off) = make_uint2(h01, h23);
        } else if (rb.accumulate_f32) {
            float* o = reinterpret_cast<float*>(job.out) + static_cast<long long>(i) * job.ldo + j;
#pragma unroll
            for (int e = 0; e < 4; ++e)
                if (e < valid) o[e] += v[e];
        } else {
            __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(job.out) + static_cast<long long>(i) * job.ldo + j;
            if (valid == 4 && ((reinterpret_cast<uintptr_t>(o) & 7) == 0)) {
                *reinterpret_cast<uint2*>(o) = make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (e < valid) o[e] = __float2bfloat16_rn(v[e]);
            }
        }
    }
}

// ------------------------------------------------ tail reduction
// Every element of a split tail tile is the sum, in piece order, of its
// pieces' partial slots: one thread per 4 consecutive columns of one row,
// bf16 store of the columns inside the output.  The slots are loaded
// TAIL_BATCH at a time ahead of their adds (a tile of a small launch has up to
// 8 pieces; loaded one after another the launch took ~6.5 us at the 2048-token
// LLaMA-60M shapes), and added in piece order, so the sums stay the same.
constexpr int TAIL_BATCH = 8;

__global__ void __launch_bounds__(RED_THREADS) tail_reduce_kernel(const __grid_constant__ TailReduce r)
{
    grid_dependency_wait();            // the partials come from the GEMM launched just before
    grid_launch_dependents();
    const int groups_per_row = r.tile_cols / 4;
    const long long per_tile = static_cast<long long>(r.tile_rows) * groups_per_row;
    const long long total = per_tile * r.ntiles;
    const long long slot_elems = static_cast<long long>(r.tile_rows) * r.tile_cols;
    const long long stride = static_cast<long long>(gridDim.x) * RED_THREADS;
    for (long long e = static_cast<long long>(blockIdx.x) * RED_THREADS + threadIdx.x; e < total; e += stride) {
        const int k = static_cast<int>(e / per_tile);
        const int local = static_cast<int>(e - static_cast<long long>(k) * per_tile);
        const int i = local / groups_per_row;
        const int j = (local - i * groups_per_row) * 4;
        const TailTile& t = r.tile[k];
        const int row = t.m0 + i, col = t.n0 + j;
        if (row >= r.M[t.g] || col >= r.N[t.g]) continue;
        const float* src = r.part + static_cast<long long>(i) * r.tile_cols + j + t.lo_slot * slot_elems;
        float4 acc = __ldg(reinterpret_cast<const float4*>(src));
        for (int q0 = 1; q0 < t.count; q0 += TAIL_BATCH) {
            float4 v[TAIL_BATCH];
#pragma unroll
            for (int b = 0; b < TAIL_BATCH; ++b)
                if (q0 + b < t.count) v[b] = __ldg(reinterpret_cast<const float4*>(src + (q0 + b) * slot_elems));
#pragma unroll
            for (int b = 0; b < TAIL_BATCH; ++b) {
                if (q0 + b < t.count) {
                    acc.x += v[b].x;
                    acc.y += v[b].y;
                    acc.z += v[b].z;
                    acc.w += v[b].w;
                }
            }
        }
        const float v[4] = {acc.x, acc.y, acc.z, acc.w};
        const int valid = min(4, r.N[t.g] - col);
        __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(r.out[t.g]) + static_cast<long long>(row) * r.ldo[t.g] + col;
        if (valid == 4 && ((reinterpret_cast<uintptr_t>(o) & 7) == 0)) {
            *reinterpret_cast<uint2*>(o) = make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
        } else {
#pragma unroll
            for (int e2 = 0; e2 < 4; ++e2)
                if (e2 < valid) o[e2] = __float2bfloat16_rn(v[e2]);
        }
    }
}

cudaError_t launch_tail_reduce(const TailReduce& r, int sms, cudaStream_t stream)
{
    const long long groups = static_cast<long long>(r.ntiles) * r.tile_rows * (r.tile_cols / 4);
    long long blocks = (groups + RED_THREADS - 1) / RED_THREADS;
    if (blocks > 8LL * sms) blocks = 8LL * sms;
    if (blocks < 1) blocks = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(RED_THREADS);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tail_reduce_kernel, r);
}

// bf16 weight gradients with a split tail (every tile configuration the planner picks)
template cudaError_t launch_gemm<128, 1, true, true, EPI_TAIL>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_TAIL>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, true, true, EPI_TAIL>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_TAIL, true>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
// split-K output GEMMs of small launches (both operands K-major)
template cudaError_t launch_gemm<128, 1, false, false, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, false, false, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, true, true, EPI_STORE>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_STORE, true>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 1, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<128, 2, true, true, EPI_F32>(const GemmBatch&, int, bool, cudaStream_t);
template cudaError_t launch_gemm<256, 1, true, true, EPI_F32, true>(const GemmBatch&, int, bool, cudaStream_t);

cudaError_t launch_splitk_reduce(ReduceBatch& rb, cudaStream_t stream)
{
    long long groups = 0;
    for (int j = 0; j < rb.count; ++j) {
        rb.job[j].group_begin = groups;
        groups += static_cast<long long>(rb.job[j].M) * ((rb.job[j].N + 3) / 4);
    }
    rb.groups = groups;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        sms = 152;
    long long blocks = (groups + RED_THREADS - 1) / RED_THREADS;
    if (blocks > 8LL * sms) blocks = 8LL * sms;   // grid-stride beyond 8 CTAs per SM
    if (blocks < 1) blocks = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(blocks));
    cfg.blockDim = dim3(RED_THREADS);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (!rb.zh) return cudaLaunchKernelEx(&cfg, splitk_reduce_kernel<false, SIG_IDENTITY>, rb);
    switch (rb.sigma) {
    case SIG_SILU: return cudaLaunchKernelEx(&cfg, splitk_reduce_kernel<true, SIG_SILU>, rb);
    case SIG_GELU: return cudaLaunchKernelEx(&cfg, splitk_reduce_kernel<true, SIG_GELU>, rb);
    case SIG_IDENTITY: return cudaLaunchKernelEx(&cfg, splitk_reduce_kernel<true, SIG_IDENTITY>, rb);
    default: return cudaErrorInvalidValue;
    }
}

}  // namespace cola
