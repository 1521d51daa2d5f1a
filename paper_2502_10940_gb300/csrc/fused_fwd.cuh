// fused_fwd.cuh -- the whole forward of one CoLA layer in one persistent
// kernel (sm_103a), for ranks r <= 128:
//
//   Z = X A^T,   H = bf16(sigma(bf16 Z)),   Y = H B^T           (Sec. 3.2, Eq. main-fwd)
//
// H is an intermediate of h = B sigma(A x), not an output: each CTA keeps
// the H of its 128-row tile in shared memory, written by the epilogue in the
// layout the tensor cores read (K-major, 128-byte swizzle), and the second
// product takes it from there.  Z and H go to global memory only when the
// mode saves them (CoLA: both, CoLA-M: Z, inference: neither).  One launch
// replaces the Z/H GEMM and the Y GEMM of the layer: no H round trip through
// HBM, one pipeline fill and one tail instead of two.  It serves launches of
// at most one 128-row tile per SM (a few thousand tokens), where a tile's
// serial Z -> H -> Y chain costs less than a second launch; the Y blocks of
// a tile are then shared by several CTAs (work items), each recomputing the
// tile's Z.  With several tiles per SM the two pipelined GEMMs were faster
// (measured: 5-13 % at 65536 tokens), and cola_fwd keeps them there.
//
// Warp roles (320 threads, one CTA per SM, persistent over work items):
//   warp 0      TMA producer: per tile, the (X, A) k-blocks of the first
//               product, then the B k-blocks of every 128-column block of Y,
//               through one ring of stages.
//   warp 1      MMA issuer: Z into TMEM columns [0, R); after the epilogue
//               has written H, each 128-column block of Y into one of two
//               accumulators (columns 128 and 256), so that the epilogue of
//               one block overlaps the MMAs of the next; allocates TMEM.
//   warps 2..9  epilogue, two warps per TMEM lane quarter taking alternate
//               32-column chunks: Z and H (stores, sigma, H into shared
//               memory), then the Y blocks (TMA stores through 32 x 32 boxes;
//               masked direct stores on a ragged right edge).
// The MMAs of item i+1's first product run while the epilogue stores item
// i's Y.  Every wait is bounded as in gemm.cuh.
#pragma once
#include "gemm.cuh"

namespace cola {

constexpr int FBN = 128;   // columns of one Y block (two double-buffered accumulators fit TMEM beside Z)

struct FusedFwdParams {
    CUtensorMap map_x;      // X [n x d_in], K-major, box {64, 128}
    CUtensorMap map_a;      // A [R x d_in], K-major, box {64, R}
    CUtensorMap map_b;      // B [d_out x R], K-major, box {64, FBN}
    CUtensorMap map_z;      // Z [n x R], 32 x 32 store boxes
    CUtensorMap map_h;      // H [n x R], 32 x 32 store boxes
    CUtensorMap map_y;      // Y [n x d_out], 32 x 32 store boxes
    int n, d_out;           // tokens, output width
    int kb1;                // k-blocks of the first product: ceil(d_in / 64)
    int m_tiles, n_blocks;  // 128-row tiles, FBN-column blocks of Y
    // work items: tile t = item / y_groups; item g = item % y_groups computes
    // Y blocks [g * blocks_per_group, +blocks_per_group) of that tile, after
    // the tile's Z (which every item of the tile recomputes; only g = 0
    // stores Z and H)
    int y_groups, blocks_per_group;
    int store_z, store_h;   // the rank-r activations the mode saves
    int sigma;
    __nv_bfloat16* y_ptr;   // Y, for the masked stores of a ragged right edge (d_out % 8 != 0)
    long long y_ld;
    unsigned int* status;
};

template <int R>
struct FusedCfg {
    static_assert(R == 64 || R == 128, "the rank of the fused forward is 64 or 128");
    static constexpr int X_BYTES = BM * BK * 2;            // one k-block of the tile's X
    static constexpr int A_BYTES = R * BK * 2;             // one k-block of A
    static constexpr int B_BYTES = FBN * BK * 2;           // one k-block of a Y block's B
    static constexpr int STAGE_BYTES = (X_BYTES + A_BYTES) > B_BYTES ? (X_BYTES + A_BYTES) : B_BYTES;
    static constexpr int H_BYTES = BM * R * 2;             // R / 64 swizzled k-blocks of 128 x 64
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM_LIMIT = 232448;
    static constexpr int STAGES_FIT = (SMEM_LIMIT - 1024 - BAR_BYTES - EPI_SMEM_BYTES - H_BYTES) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + H_BYTES + EPI_SMEM_BYTES + BAR_BYTES;
    static_assert(SMEM_BYTES <= SMEM_LIMIT, "shared memory budget");
    static_assert(STAGES >= 3, "a useful ring");
    static constexpr int TMEM_COLS = 512;                  // Z at 0, Y blocks at 128 and 256
    static constexpr int Y_COL0 = 128;
};

template <int R>
__global__ void __launch_bounds__(NUM_THREADS, 1) fused_fwd_kernel(const __grid_constant__ FusedFwdParams P)
{
    using C = FusedCfg<R>;
    constexpr int STAGES = C::STAGES;
    constexpr int KH = R / BK;                 // k-blocks of the second product
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;                                       // STAGES x STAGE_BYTES
    uint8_t* hbuf = smem + STAGES * C::STAGE_BYTES;             // H of the tile in hand
    uint8_t* smem_epi = hbuf + C::H_BYTES;                      // NUM_EPI_WARPS x EPI_WARP_BYTES
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem_epi + EPI_SMEM_BYTES);
    uint64_t* full_bar = bars;                 // [STAGES]
    uint64_t* empty_bar = bars + STAGES;       // [STAGES]
    uint64_t* zfull = bars + 2 * STAGES;       // Z accumulated (MMA commit)
    uint64_t* zempty = zfull + 1;              // Z read by the epilogue
    uint64_t* hfull = zempty + 1;              // H written to shared memory by the epilogue
    uint64_t* hempty = hfull + 1;              // the MMAs that read H are done (MMA commit)
    uint64_t* yfull = hempty + 1;              // [2] a Y block accumulated
    uint64_t* yempty = yfull + 2;              // [2] a Y block read by the epilogue
    uint64_t* drain_bar = yempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const WaitCtx wc{abort_flag, P.status};
    constexpr int EPI_THREADS = NUM_EPI_WARPS * 32;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        mbar_init(zfull, 1);
        mbar_init(zempty, EPI_THREADS);
        mbar_init(hfull, EPI_THREADS);
        mbar_init(hempty, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&yfull[b], 1);
            mbar_init(&yempty[b], EPI_THREADS);
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&P.map_x);
        tma_prefetch_desc(&P.map_a);
        tma_prefetch_desc(&P.map_b);
        tma_prefetch_desc(&P.map_y);
        if (P.store_z) tma_prefetch_desc(&P.map_z);
        if (P.store_h) tma_prefetch_desc(&P.map_h);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    grid_dependency_wait();
    grid_launch_dependents();

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            long long issued = 0;
            bool ok = true;
            auto next = [&]() {
                ++issued;
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            };
            for (int item = blockIdx.x; item < P.m_tiles * P.y_groups && ok; item += gridDim.x) {
                const int m0 = (item / P.y_groups) * BM;
                const int nb0 = (item % P.y_groups) * P.blocks_per_group;
                const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
                for (int kb = 0; kb < P.kb1 && ok; ++kb) {
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t* st = ring + stage * C::STAGE_BYTES;
                    mbar_arrive_expect_tx(&full_bar[stage], C::X_BYTES + C::A_BYTES);
                    tma_load_2d(&P.map_x, &full_bar[stage], st, kb * BK, m0);
                    tma_load_2d(&P.map_a, &full_bar[stage], st + C::X_BYTES, kb * BK, 0);
                    next();
                }
                for (int nb = nb0; nb < nb1 && ok; ++nb) {
                    for (int k2 = 0; k2 < KH; ++k2) {
                        if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        uint8_t* st = ring + stage * C::STAGE_BYTES;
                        mbar_arrive_expect_tx(&full_bar[stage], C::B_BYTES);
                        tma_load_2d(&P.map_b, &full_bar[stage], st, k2 * BK, nb * FBN);
                        next();
                    }
                }
            }
            bool normal = ok && !*abort_flag;
            const int stage_end = stage;
            const uint32_t phase_end = phase;
            if (normal) {
                for (int j = 0; j < STAGES; ++j) {   // every stage released by the MMA warp
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        normal = false;
                        break;
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!normal) {   // drain: the last min(issued, STAGES) loads may still be landing
                const int outstanding = issued < STAGES ? static_cast<int>(issued) : STAGES;
                int s = stage_end;
                uint32_t ph = phase_end;
                for (int j = 0; j < outstanding; ++j) {
                    if (--s < 0) {
                        s = STAGES - 1;
                        ph ^= 1u;
                    }
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(&full_bar[s], ph)) {
                        if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                            if (P.status) atomicOr(P.status, ST_TIMEOUT_DRAIN);
                            break;
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_z = idesc_bf16_f32(BM, R, 0, 0);
            constexpr uint32_t idesc_y = idesc_bf16_f32(BM, FBN, 0, 0);
            const uint32_t h_addr = smem_u32(hbuf);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true, issued_any = false;
            long long yblk = 0;   // Y blocks issued so far: buffer yblk & 1, use (yblk >> 1)
            auto next = [&]() {
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            };
            int it = 0;
            for (int item = blockIdx.x; item < P.m_tiles * P.y_groups && ok; item += gridDim.x, ++it) {
                const uint32_t par = static_cast<uint32_t>(it & 1);
                const int nb0 = (item % P.y_groups) * P.blocks_per_group;
                const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
                // first product: Z = X A^T
                if (!wait_bounded(zempty, par ^ 1u, wc, ST_TIMEOUT_MMA)) break;
                tc_fence_after();
                for (int kb = 0; kb < P.kb1; ++kb) {
                    if (!wait_bounded(&full_bar[stage], phase, wc, ST_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sx = smem_u32(ring + stage * C::STAGE_BYTES);
#pragma unroll
                    for (int ks = 0; ks < BK / UMMA_K; ++ks)
                        umma_f16(tmem_base, smem_desc_sw128(sx + ks * UMMA_K * 2, 16, 1024),
                                 smem_desc_sw128(sx + C::X_BYTES + ks * UMMA_K * 2, 16, 1024), idesc_z,
                                 (kb > 0 || ks > 0) ? 1u : 0u);
                    issued_any = true;
                    umma_commit(&empty_bar[stage]);
                    next();
                }
                if (!ok) break;
                umma_commit(zfull);
                // second product: Y = H B^T, once the epilogue has written H
                if (!wait_bounded(hfull, par, wc, ST_TIMEOUT_MMA)) break;
                tc_fence_after();
                for (int nb = nb0; nb < nb1 && ok; ++nb, ++yblk) {
                    const int b = static_cast<int>(yblk & 1);
                    const uint32_t ypar = static_cast<uint32_t>((yblk >> 1) & 1);
                    if (!wait_bounded(&yempty[b], ypar ^ 1u, wc, ST_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d_y = tmem_base + static_cast<uint32_t>(C::Y_COL0 + b * FBN);
                    for (int k2 = 0; k2 < KH; ++k2) {
                        if (!wait_bounded(&full_bar[stage], phase, wc, ST_TIMEOUT_MMA)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t sb = smem_u32(ring + stage * C::STAGE_BYTES);
                        const uint32_t sh = h_addr + k2 * (BM * BK * 2);
#pragma unroll
                        for (int ks = 0; ks < BK / UMMA_K; ++ks)
                            umma_f16(d_y, smem_desc_sw128(sh + ks * UMMA_K * 2, 16, 1024),
                                     smem_desc_sw128(sb + ks * UMMA_K * 2, 16, 1024), idesc_y,
                                     (k2 > 0 || ks > 0) ? 1u : 0u);
                        umma_commit(&empty_bar[stage]);
                        next();
                    }
                    if (!ok) break;
                    umma_commit(&yfull[b]);
                }
                if (!ok) break;
                umma_commit(hempty);   // H may be overwritten once these MMAs are done
            }
            if ((!ok || *abort_flag) && issued_any) {
                umma_commit(drain_bar);
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0)) {
                    if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                        if (P.status) atomicOr(P.status, ST_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..9)
        const int q = warp & 3;                 // TMEM lane quarter
        const int half = (warp - 2) >> 2;       // alternate 32-column chunks
        const int row_in = q * 32 + lane;       // this thread's row of the tile
        const uint32_t ep = smem_u32(smem_epi + (warp - 2) * EPI_WARP_BYTES);
        const uint32_t h_addr = smem_u32(hbuf);
        int out_slot = 0;
        long long yblk = 0;

        auto emit = [&](const CUtensorMap* map, const uint32_t (&w)[16], int x, int y) {
            if (y >= P.n) return;               // the whole box lies below the last token
            const uint32_t box = ep + out_slot * EPI_BOX_BYTES;
            if (lane == 0) bulk_wait_group_read<EPI_OUT_BOXES - 1>();
            __syncwarp();
            stage_row(box, lane, w);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                tma_store_2d(map, box, x, y);
                bulk_commit_group();
            }
            if (++out_slot == EPI_OUT_BOXES) out_slot = 0;
        };

        int it = 0;
        for (int item = blockIdx.x; item < P.m_tiles * P.y_groups; item += gridDim.x, ++it) {
            const uint32_t par = static_cast<uint32_t>(it & 1);
            const int row0 = (item / P.y_groups) * BM + q * 32;    // first row of this warp's 32
            const bool first = item % P.y_groups == 0;             // the item that stores Z and H
            const int nb0 = (item % P.y_groups) * P.blocks_per_group;
            const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
            // ---- Z, H = sigma(Z): global stores as the mode saves them; H into shared memory
            if (!wait_bounded(zfull, par, wc, ST_TIMEOUT_EPILOGUE)) break;
            if (!wait_bounded(hempty, par ^ 1u, wc, ST_TIMEOUT_EPILOGUE)) break;
            tc_fence_after();
            for (int c = half; c < R / 32; c += 2) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + c * 32, v);
                tmem_ld_wait();
                uint32_t w[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                if (P.store_z && first) emit(&P.map_z, w, c * 32, row0);
                with_sigma(P.sigma, [&](auto tag) {
                    constexpr int S = decltype(tag)::value;
#pragma unroll
                    for (int j = 0; j < 16; ++j) w[j] = pack_bf16x2(act_sigma<S>(bf16_lo(w[j])), act_sigma<S>(bf16_hi(w[j])));
                });
                if (P.store_h && first) emit(&P.map_h, w, c * 32, row0);
                // H row `row_in`, columns c*32 .. c*32+31: k-block c / 2, 16-byte chunks
                // 4 (c & 1) .. +3 of the 128-byte row, swizzled by the row's position in its 8-row group
                const uint32_t rbase = h_addr + (c >> 1) * (BM * BK * 2) + row_in * 128;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int chunk = 4 * (c & 1) + j;
                    st_shared_v4(rbase + ((chunk ^ (row_in & 7)) << 4), w[4 * j], w[4 * j + 1], w[4 * j + 2],
                                 w[4 * j + 3]);
                }
            }
            tc_fence_before();
            mbar_arrive(zempty);                // Z read: the next tile's first product may start
            fence_proxy_async_smem();           // H visible to the tensor cores
            mbar_arrive(hfull);
            // ---- Y blocks
            bool ok = true;
            for (int nb = nb0; nb < nb1; ++nb, ++yblk) {
                const int b = static_cast<int>(yblk & 1);
                if (!wait_bounded(&yfull[b], static_cast<uint32_t>((yblk >> 1) & 1), wc, ST_TIMEOUT_EPILOGUE)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int left = P.d_out - nb * FBN;
                const int nch = row0 >= P.n ? 0 : (left >= FBN ? FBN / 32 : (left + 31) / 32);
                for (int c = half; c < nch; c += 2) {
                    const int col0 = nb * FBN + c * 32;
                    uint32_t v[32];
                    tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                           static_cast<uint32_t>(C::Y_COL0 + b * FBN + c * 32), v);
                    tmem_ld_wait();
                    uint32_t w[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    if ((P.d_out & 7) != 0 && col0 + 32 > P.d_out) {
                        // ragged right edge: masked per-element stores, padding untouched
                        const int row = row0 + lane;
                        if (row < P.n) {
                            uint16_t* d = reinterpret_cast<uint16_t*>(P.y_ptr + row * P.y_ld + col0);
                            const int valid = P.d_out - col0;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (j < valid) d[j] = static_cast<uint16_t>((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xFFFFu));
                        }
                        continue;
                    }
                    emit(&P.map_y, w, col0, row0);
                }
                tc_fence_before();
                mbar_arrive(&yempty[b]);
            }
            if (!ok) break;
        }
        if (lane == 0) bulk_wait_group_all();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

}  // namespace cola
