// gemm.cuh -- the one tensor-core GEMM every CoLA step runs on (sm_103a).
//
//   D[M x N] = sum_k  Aop[m, k] * Bop[n, k]        (fp32 accumulation in TMEM)
//
// Each operand lives in global memory either K-major (k contiguous, the
// nn.Linear weight layout) or MN-major (m / n contiguous, a token-major
// activation read "transposed").  Both are staged by TMA into 128-byte
// swizzled shared memory and consumed by tcgen05.mma directly, so no
// operand is ever transposed in memory.
//
// Warp roles (192 threads, one CTA per SM, persistent over output tiles):
//   warp 0      TMA producer: fills a STAGES-deep ring of (A, B) k-blocks.
//   warp 1      MMA issuer:  tcgen05.mma M=128, N=BN, K=16 into one of two
//               TMEM accumulators (double buffered, so the epilogue of tile
//               i overlaps the main loop of tile i+1); allocates TMEM.
//   warps 2..5  epilogue: tcgen05.ld -> fused elementwise -> global stores.
//
// Epilogues (the elementwise parts of the layer, fused so that the rank-r
// intermediate makes no extra HBM round trip):
//   EPI_STORE   D = bf16(acc)                                  (Y, dX)
//   EPI_ZH      Z = bf16(acc), H = bf16(sigma(Z))              (forward A-GEMM)
//   EPI_DSIGMA  dZ = bf16(acc * sigma'(Z_saved)); with CoLA-M also
//               H = bf16(sigma(Z_saved)) for the weight gradient of B
//   EPI_F32     fp32 split-K partial slab (weight gradients, reduced later)
//
// Every mbarrier wait is bounded (WAIT_LIMIT_NS of global time).  On expiry
// the waiting thread records where it gave up in the status word, raises a
// CTA-wide abort flag that makes every other wait return, waits (bounded) for
// its own copies and MMAs still in flight, and the CTA frees its TMEM and
// exits.  No wait can spin forever.
#pragma once
#include <cuda_bf16.h>
#include <cstdint>

#include "ptx.cuh"

namespace cola {

constexpr int BM = 128;              // UMMA M (cta_group::1): one row per TMEM lane
constexpr int BK = 64;               // k-block: one 128-byte swizzle row of bf16
constexpr int UMMA_K = 16;           // K of one kind::f16 MMA
constexpr int NUM_THREADS = 192;
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;   // 2 s

// bits recorded in the status word when a wait gives up
enum : unsigned int {
    ST_TIMEOUT_PRODUCER = 1u << 0,
    ST_TIMEOUT_MMA = 1u << 1,
    ST_TIMEOUT_EPILOGUE = 1u << 2,
    ST_TIMEOUT_DRAIN = 1u << 3,
};

enum Epi : int { EPI_STORE = 0, EPI_ZH = 1, EPI_DSIGMA = 2, EPI_F32 = 3 };
enum Sigma : int { SIG_IDENTITY = 0, SIG_SILU = 1, SIG_GELU = 2 };

struct GemmParams {
    int M, N;              // logical output extents
    int k_blocks;          // ceil(K / BK)
    int m_tiles, n_tiles;
    int splits, kb_per_split;
    int units;             // m_tiles * n_tiles * splits
    void* D;               // bf16 output, or fp32 partial slabs (EPI_F32)
    long long ldd;         // row pitch of D in elements
    __nv_bfloat16* D2;     // H output (EPI_ZH / EPI_DSIGMA), may be null
    long long ldd2;
    const __nv_bfloat16* Zin;  // saved Z (EPI_DSIGMA)
    long long ldz;
    long long part_stride; // EPI_F32: elements per split slab
    int sigma;
    unsigned int* status;
};

template <int BN>
struct GemmCfg {
    static_assert(BN % 64 == 0 && BN >= 64 && BN <= 256, "BN must be 64..256 in steps of 64");
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGES = (200 * 1024) / STAGE_BYTES > 8 ? 8 : (200 * 1024) / STAGE_BYTES;
    static constexpr int TMEM_COLS = (2 * BN <= 128) ? 128 : (2 * BN <= 256 ? 256 : 512);
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + BAR_BYTES;
};

// ------------------------------------------------------------ activations
__device__ __forceinline__ float act_sigma(int kind, float z)
{
    if (kind == SIG_SILU) return z / (1.0f + __expf(-z));
    if (kind == SIG_GELU) return 0.5f * z * erfcf(-z * 0.70710678118654752f);
    return z;
}

__device__ __forceinline__ float act_dsigma(int kind, float z)
{
    if (kind == SIG_SILU) {
        const float s = 1.0f / (1.0f + __expf(-z));
        return s * (1.0f + z * (1.0f - s));
    }
    if (kind == SIG_GELU) {
        const float Phi = 0.5f * erfcf(-z * 0.70710678118654752f);
        const float phi = 0.39894228040143268f * __expf(-0.5f * z * z);
        return Phi + z * phi;
    }
    return 1.0f;
}

// --------------------------------------------------------- bounded waits
struct WaitCtx {
    volatile int* abort_flag;
    unsigned int* status;
};

__device__ __forceinline__ bool wait_bounded(uint64_t* bar, uint32_t parity, const WaitCtx& w, unsigned int code)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*w.abort_flag) return false;
        if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
            *w.abort_flag = 1;
            if (w.status) atomicOr(w.status, code);
            return false;
        }
    }
}

__device__ __forceinline__ void decode_unit(const GemmParams& p, int u, int& m_blk, int& n_blk, int& split,
                                            int& kb0, int& kb1)
{
    const int tiles = p.m_tiles * p.n_tiles;
    split = u / tiles;
    const int rem = u - split * tiles;
    m_blk = rem / p.n_tiles;
    n_blk = rem - m_blk * p.n_tiles;
    kb0 = split * p.kb_per_split;
    kb1 = min(kb0 + p.kb_per_split, p.k_blocks);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Store 32 packed bf16 (16 words) at dst[0..31], clipped to `valid` columns.
__device__ __forceinline__ void store_row32_bf16(__nv_bfloat16* dst, const uint32_t (&w)[16], int valid)
{
    if (valid >= 32) {
        uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int q = 0; q < 4; ++q) d4[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
    } else {
        uint16_t* d = reinterpret_cast<uint16_t*>(dst);
        for (int j = 0; j < valid; ++j) d[j] = static_cast<uint16_t>((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xFFFFu));
    }
}

// ------------------------------------------------------------ the kernel
template <int BN, bool A_MN, bool B_MN, int EPI>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b,
                const GemmParams p)
{
    using C = GemmCfg<BN>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* smem_a = smem;                              // STAGES x A_BYTES
    uint8_t* smem_b = smem + STAGES * C::A_BYTES;        // STAGES x B_BYTES
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * C::STAGE_BYTES);
    uint64_t* full_bar = bars;                 // [STAGES]
    uint64_t* empty_bar = bars + STAGES;       // [STAGES]
    uint64_t* tfull_bar = bars + 2 * STAGES;   // [2]
    uint64_t* tempty_bar = tfull_bar + 2;      // [2]
    uint64_t* drain_bar = tempty_bar + 2;      // [1]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const WaitCtx wc{abort_flag, p.status};

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull_bar[b], 1);
            mbar_init(&tempty_bar[b], 4 * 32);
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&map_a);
        tma_prefetch_desc(&map_b);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            long long issued = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
                int m_blk, n_blk, split, kb0, kb1;
                decode_unit(p, u, m_blk, n_blk, split, kb0, kb1);
                const int m0 = m_blk * BM, n0 = n_blk * BN;
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sa = smem_a + stage * C::A_BYTES;
                    uint8_t* sb = smem_b + stage * C::B_BYTES;
                    mbar_arrive_expect_tx(&full_bar[stage], C::STAGE_BYTES);
                    const int k0 = kb * BK;
                    if (A_MN) {
                        tma_load_2d(&map_a, &full_bar[stage], sa, m0, k0);
                        tma_load_2d(&map_a, &full_bar[stage], sa + 64 * BK * 2, m0 + 64, k0);
                    } else {
                        tma_load_2d(&map_a, &full_bar[stage], sa, k0, m0);
                    }
                    if (B_MN) {
#pragma unroll
                        for (int j = 0; j < BN / 64; ++j)
                            tma_load_2d(&map_b, &full_bar[stage], sb + j * 64 * BK * 2, n0 + 64 * j, k0);
                    } else {
                        tma_load_2d(&map_b, &full_bar[stage], sb, k0, n0);
                    }
                    ++issued;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (ok && !*abort_flag) {
                // tail: acquire every stage once more, i.e. wait until the MMA warp
                // has released (its commits have arrived on) all of them
                for (int j = 0; j < STAGES; ++j) {
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) break;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            } else {
                // drain: the last min(issued, STAGES) loads may still be landing
                const int outstanding = issued < STAGES ? static_cast<int>(issued) : STAGES;
                int s = stage;
                uint32_t ph = phase;
                for (int j = 0; j < outstanding; ++j) {
                    if (--s < 0) {
                        s = STAGES - 1;
                        ph ^= 1u;
                    }
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(&full_bar[s], ph)) {
                        if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                            if (p.status) atomicOr(p.status, ST_TIMEOUT_DRAIN);
                            break;
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
            int stage = 0;
            uint32_t phase = 0;
            int buf = 0;
            uint32_t bphase = 0;
            bool ok = true;
            bool issued_any = false;
            for (int u = blockIdx.x; u < p.units && ok; u += gridDim.x) {
                int m_blk, n_blk, split, kb0, kb1;
                decode_unit(p, u, m_blk, n_blk, split, kb0, kb1);
                if (!wait_bounded(&tempty_bar[buf], bphase ^ 1u, wc, ST_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!wait_bounded(&full_bar[stage], phase, wc, ST_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(smem_a + stage * C::A_BYTES);
                    const uint32_t sb = smem_u32(smem_b + stage * C::B_BYTES);
#pragma unroll
                    for (int ks = 0; ks < BK / UMMA_K; ++ks) {
                        // K-major: next 16 k = +32 bytes inside the swizzled 128-byte row.
                        // MN-major: next 16 k = +16 rows of 128 bytes.
                        const uint64_t da = A_MN ? smem_desc_sw128(sa + ks * UMMA_K * 128, 64 * BK * 2, 1024)
                                                 : smem_desc_sw128(sa + ks * UMMA_K * 2, 16, 1024);
                        const uint64_t db = B_MN ? smem_desc_sw128(sb + ks * UMMA_K * 128, 64 * BK * 2, 1024)
                                                 : smem_desc_sw128(sb + ks * UMMA_K * 2, 16, 1024);
                        umma_f16(d_tmem, da, db, idesc, (kb > kb0 || ks > 0) ? 1u : 0u);
                    }
                    issued_any = true;
                    umma_commit(&empty_bar[stage]);   // frees the smem stage once these MMAs are done
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(&tfull_bar[buf]);         // accumulator ready for the epilogue
                if (++buf == 2) {
                    buf = 0;
                    bphase ^= 1u;
                }
            }
            if ((!ok || *abort_flag) && issued_any) {
                umma_commit(drain_bar);
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0)) {
                    if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                        if (p.status) atomicOr(p.status, ST_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        const int q = warp & 3;                 // TMEM lane quarter this warp may access
        const int row_in_tile = q * 32 + lane;
        int buf = 0;
        uint32_t bphase = 0;
        for (int u = blockIdx.x; u < p.units; u += gridDim.x) {
            int m_blk, n_blk, split, kb0, kb1;
            decode_unit(p, u, m_blk, n_blk, split, kb0, kb1);
            if (!wait_bounded(&tfull_bar[buf], bphase, wc, ST_TIMEOUT_EPILOGUE)) break;
            tc_fence_after();
            const int row = m_blk * BM + row_in_tile;
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(buf * BN);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tbase + c * 32, v);
                tmem_ld_wait();
                const int col0 = n_blk * BN + c * 32;
                if (EPI == EPI_F32) {
                    float* dst = reinterpret_cast<float*>(p.D) + split * p.part_stride +
                                 static_cast<long long>(m_blk * BM + row_in_tile) * (p.n_tiles * BN) + col0;
                    float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        d4[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                            __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    continue;
                }
                if (row >= p.M || col0 >= p.N) continue;
                const int valid = min(32, p.N - col0);
                uint32_t w[16];
                if (EPI == EPI_STORE) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    store_row32_bf16(reinterpret_cast<__nv_bfloat16*>(p.D) + row * p.ldd + col0, w, valid);
                } else if (EPI == EPI_ZH) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    store_row32_bf16(reinterpret_cast<__nv_bfloat16*>(p.D) + row * p.ldd + col0, w, valid);
                    if (p.D2 != nullptr) {
                        uint32_t h[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            h[j] = pack_bf16x2(act_sigma(p.sigma, bf16_lo(w[j])), act_sigma(p.sigma, bf16_hi(w[j])));
                        store_row32_bf16(p.D2 + row * p.ldd2 + col0, h, valid);
                    }
                } else if (EPI == EPI_DSIGMA) {
                    // Z has the same (row, col) extent as dZ: N = r is a multiple of 64.
                    uint32_t z[16];
                    const uint4* zs = reinterpret_cast<const uint4*>(p.Zin + row * p.ldz + col0);
#pragma unroll
                    for (int qd = 0; qd < 4; ++qd) {
                        const uint4 t = zs[qd];
                        z[4 * qd] = t.x;
                        z[4 * qd + 1] = t.y;
                        z[4 * qd + 2] = t.z;
                        z[4 * qd + 3] = t.w;
                    }
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float z0 = bf16_lo(z[j]), z1 = bf16_hi(z[j]);
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]) * act_dsigma(p.sigma, z0),
                                           __uint_as_float(v[2 * j + 1]) * act_dsigma(p.sigma, z1));
                    }
                    store_row32_bf16(reinterpret_cast<__nv_bfloat16*>(p.D) + row * p.ldd + col0, w, valid);
                    if (p.D2 != nullptr) {
                        uint32_t h[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            h[j] = pack_bf16x2(act_sigma(p.sigma, bf16_lo(z[j])), act_sigma(p.sigma, bf16_hi(z[j])));
                        store_row32_bf16(p.D2 + row * p.ldd2 + col0, h, valid);
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&tempty_bar[buf]);
            if (++buf == 2) {
                buf = 0;
                bphase ^= 1u;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

}  // namespace cola
