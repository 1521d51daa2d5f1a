// fused_layer.cuh -- one pass of a CoLA layer with r <= 128 in one persistent
// kernel (sm_103a): two chained products whose rank-r intermediate never
// leaves the chip.
//
//   forward  (BWD = false):  Z  = X A^T,  H = bf16(sigma(bf16 Z)),      Y  = H B^T   (Sec. 3.2, Eq. main-fwd)
//   backward (BWD = true):   dZ = bf16((dY B) * sigma'(Z_saved)),       dX = dZ A    (Sec. 3.4: dH = dY B,
//                                                                                     the chain rule through sigma)
//
// H (forward) and dZ (backward) are intermediates of the layer's pass, not
// its outputs: each CTA keeps the one of its 128-row tile in shared memory,
// written by the epilogue in the layout the tensor cores read (K-major,
// 128-byte swizzle), and the second product takes it from there.
//   forward   Z and H go to global memory only when the mode saves them
//             (CoLA: both, CoLA-M: Z, inference: neither).
//   backward  the tile's saved Z is TMA-loaded into that same buffer; the
//             epilogue reads each row's Z from it, multiplies the first
//             product by sigma'(Z) and writes dZ in Z's place.  dZ always
//             goes to global memory too (the weight gradient dA = dZ^T X
//             reads it), and so does H = sigma(Z) under CoLA-M (dB = dY^T H
//             reads it).
// One launch replaces the two GEMMs of the pass: no intermediate round trip
// through HBM, one pipeline fill and one tail instead of two.  It serves
// launches of at most one 128-row tile per SM (a few thousand tokens), where
// a tile's serial chain (first product -> epilogue -> second product) costs
// less than a second launch; the 128-column output blocks of a tile are then
// shared by several CTAs (work items), each recomputing the tile's first
// product.  With several tiles per SM the two pipelined GEMMs were faster
// (forward, measured: 5-13 % at 65536 tokens), and the host keeps them there.
//
// Operands: the first product's A operand (X / dY) is token-major, K-major.
// Its B operand (A / B) and the second product's B operand (B / A) are the
// layer's weights: K-major in the forward (nn.Linear layout), MN-major in the
// backward (the same weights read transposed), staged as 64 x 64 boxes.
//
// Warp roles (320 threads, one CTA per SM, persistent over work items):
//   warp 0      TMA producer: per item, the k-blocks of the first product,
//               (backward) the tile's saved Z once the previous item's second
//               product is done with the buffer, then the weight k-blocks of
//               every output block, through one ring of stages.
//   warp 1      MMA issuer: the first product into TMEM columns [0, R); after
//               the epilogue has written the intermediate, each 128-column
//               output block into one of two accumulators (columns 128 and
//               256), so that the epilogue of one block overlaps the MMAs of
//               the next; allocates TMEM.
//   warps 2..9  epilogue, two warps per TMEM lane quarter taking alternate
//               32-column chunks: the rank-r step (stores, sigma or sigma',
//               the intermediate into shared memory), then the output blocks
//               (TMA stores through 32 x 32 boxes; masked direct stores on a
//               ragged right edge).
// The MMAs of item i+1's first product run while the epilogue stores item
// i's output.  Every wait is bounded as in gemm.cuh.
#pragma once
#include "gemm.cuh"

namespace cola {

constexpr int FBN = 128;   // columns of one output block (two double-buffered accumulators fit TMEM beside the first)

struct FusedParams {
    CUtensorMap map_in;     // first product, A operand: X [n x d_in] / dY [n x d_out], K-major, box {64, 128}
    CUtensorMap map_w1;     // first product, B operand: A [R x d_in], K-major, box {64, R} /
                            //                           B [d_out x R], MN-major, box {64, 64}
    CUtensorMap map_w2;     // second product, B operand: B [d_out x R], K-major, box {64, FBN} /
                            //                            A [R x d_in], MN-major, box {64, 64}
    CUtensorMap map_zin;    // backward: the saved Z [n x R], K-major, box {64, 128}
    CUtensorMap map_s1;     // Z / dZ [n x R], 32 x 32 store boxes
    CUtensorMap map_s2;     // H [n x R], 32 x 32 store boxes
    CUtensorMap map_out;    // Y [n x d_out] / dX [n x d_in], 32 x 32 store boxes
    int n, n_out;           // tokens, width of the second product's output
    int kb1;                // k-blocks of the first product
    int m_tiles, n_blocks;  // 128-row tiles, FBN-column output blocks
    // work items: tile t = item / out_groups; item g = item % out_groups
    // computes output blocks [g * blocks_per_group, +blocks_per_group) of
    // that tile, after the tile's first product (which every item of the
    // tile recomputes; only g = 0 stores the rank-r results)
    int out_groups, blocks_per_group;
    int store_s1, store_s2; // the rank-r results stored
    int sigma;
    __nv_bfloat16* out_ptr; // the output, for the masked stores of a ragged right edge (n_out % 8 != 0)
    long long out_ld;
    unsigned int* status;
};

template <int R>
struct FusedCfg {
    static_assert(R == 64 || R == 128, "the rank of the fused layer kernels is 64 or 128");
    static constexpr int IN_BYTES = BM * BK * 2;           // one k-block of the tile's first operand
    static constexpr int W1_BYTES = R * BK * 2;            // one k-block of the first product's weights
    static constexpr int W2_BYTES = FBN * BK * 2;          // one k-block of an output block's weights
    static constexpr int STAGE_BYTES = (IN_BYTES + W1_BYTES) > W2_BYTES ? (IN_BYTES + W1_BYTES) : W2_BYTES;
    static constexpr int T_BYTES = BM * R * 2;             // the tile's intermediate: R / 64 swizzled k-blocks of 128 x 64
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM_LIMIT = 232448;
    static constexpr int STAGES_FIT = (SMEM_LIMIT - 1024 - BAR_BYTES - EPI_SMEM_BYTES - T_BYTES) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + T_BYTES + EPI_SMEM_BYTES + BAR_BYTES;
    static_assert(SMEM_BYTES <= SMEM_LIMIT, "shared memory budget");
    static_assert(STAGES >= 3, "a useful ring");
    static constexpr int TMEM_COLS = 512;                  // first product at 0, output blocks at 128 and 256
    static constexpr int OUT_COL0 = 128;
};

// UMMA shared-memory descriptor of k-step ks (16 k) of a stage operand:
// K-major, +32 bytes inside the swizzled 128-byte row; MN-major (64 x 64
// boxes, one per 64 MN indices, 8 KB apart), +16 rows of 128 bytes.
template <bool MN>
__device__ __forceinline__ uint64_t fused_operand_desc(uint32_t base, int ks)
{
    return MN ? smem_desc_sw128(base + ks * UMMA_K * 128, 64 * BK * 2, 1024)
              : smem_desc_sw128(base + ks * UMMA_K * 2, 16, 1024);
}

template <int R, bool BWD, int SIG>
__global__ void __launch_bounds__(NUM_THREADS, 1) fused_layer_kernel(const __grid_constant__ FusedParams P)
{
    using C = FusedCfg<R>;
    constexpr int STAGES = C::STAGES;
    constexpr int KH = R / BK;                 // k-blocks of the second product
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* ring = smem;                                       // STAGES x STAGE_BYTES
    uint8_t* tbuf = smem + STAGES * C::STAGE_BYTES;             // the intermediate of the tile in hand
    uint8_t* smem_epi = tbuf + C::T_BYTES;                      // NUM_EPI_WARPS x EPI_WARP_BYTES
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem_epi + EPI_SMEM_BYTES);
    uint64_t* full_bar = bars;                 // [STAGES]
    uint64_t* empty_bar = bars + STAGES;       // [STAGES]
    uint64_t* zfull = bars + 2 * STAGES;       // first product accumulated (MMA commit)
    uint64_t* zempty = zfull + 1;              // first product read by the epilogue
    uint64_t* hfull = zempty + 1;              // intermediate written to shared memory by the epilogue
    uint64_t* hempty = hfull + 1;              // the MMAs that read the intermediate are done (MMA commit)
    uint64_t* yfull = hempty + 1;              // [2] an output block accumulated
    uint64_t* yempty = yfull + 2;              // [2] an output block read by the epilogue
    uint64_t* drain_bar = yempty + 2;
    uint64_t* zld = drain_bar + 1;             // backward: the tile's saved Z landed in tbuf
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(zld + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const WaitCtx wc{abort_flag, P.status};
    constexpr int EPI_THREADS = NUM_EPI_WARPS * 32;
    const int items = P.m_tiles * P.out_groups;

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
        mbar_init(zld, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&P.map_in);
        tma_prefetch_desc(&P.map_w1);
        tma_prefetch_desc(&P.map_w2);
        tma_prefetch_desc(&P.map_out);
        if (BWD) tma_prefetch_desc(&P.map_zin);
        if (P.store_s1) tma_prefetch_desc(&P.map_s1);
        if (P.store_s2) tma_prefetch_desc(&P.map_s2);
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
            int z_issued = 0;         // backward: Z loads issued (one per item, the i-th completing phase i of zld)
            auto next = [&]() {
                ++issued;
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            };
            int it = 0;
            for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++it) {
                const int m0 = (item / P.out_groups) * BM;
                const int nb0 = (item % P.out_groups) * P.blocks_per_group;
                const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
                for (int kb = 0; kb < P.kb1 && ok; ++kb) {
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t* st = ring + stage * C::STAGE_BYTES;
                    mbar_arrive_expect_tx(&full_bar[stage], C::IN_BYTES + C::W1_BYTES);
                    tma_load_2d(&P.map_in, &full_bar[stage], st, kb * BK, m0);
                    if (BWD) {
#pragma unroll
                        for (int j = 0; j < R / 64; ++j)
                            tma_load_2d(&P.map_w1, &full_bar[stage], st + C::IN_BYTES + j * 64 * BK * 2, 64 * j, kb * BK);
                    } else {
                        tma_load_2d(&P.map_w1, &full_bar[stage], st + C::IN_BYTES, kb * BK, 0);
                    }
                    next();
                }
                if (BWD && ok) {
                    // the tile's saved Z into tbuf, once the previous item's
                    // second product has read the dZ there
                    if (!wait_bounded(hempty, static_cast<uint32_t>(it & 1) ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(zld, C::T_BYTES);
#pragma unroll
                    for (int j = 0; j < R / 64; ++j) tma_load_2d(&P.map_zin, zld, tbuf + j * (BM * BK * 2), 64 * j, m0);
                    ++z_issued;
                }
                for (int nb = nb0; nb < nb1 && ok; ++nb) {
                    for (int k2 = 0; k2 < KH; ++k2) {
                        if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        uint8_t* st = ring + stage * C::STAGE_BYTES;
                        mbar_arrive_expect_tx(&full_bar[stage], C::W2_BYTES);
                        if (BWD) {
#pragma unroll
                            for (int j = 0; j < FBN / 64; ++j)
                                tma_load_2d(&P.map_w2, &full_bar[stage], st + j * 64 * BK * 2, nb * FBN + 64 * j, k2 * BK);
                        } else {
                            tma_load_2d(&P.map_w2, &full_bar[stage], st, k2 * BK, nb * FBN);
                        }
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
            if (BWD && z_issued > 0) {
                // the last Z load has landed before the CTA can exit, also when
                // the epilogue gave up before waiting for it (each load is issued
                // after the previous one's phase completed: hempty of the item
                // before it follows that item's zld wait)
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(zld, static_cast<uint32_t>((z_issued - 1) & 1))) {
                    if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                        if (P.status) atomicOr(P.status, ST_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc_1 = idesc_bf16_f32(BM, R, 0, BWD ? 1 : 0);
            constexpr uint32_t idesc_2 = idesc_bf16_f32(BM, FBN, 0, BWD ? 1 : 0);
            const uint32_t t_addr = smem_u32(tbuf);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true, issued_any = false;
            long long yblk = 0;   // output blocks issued so far: buffer yblk & 1, use (yblk >> 1)
            auto next = [&]() {
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            };
            int it = 0;
            for (int item = blockIdx.x; item < items && ok; item += gridDim.x, ++it) {
                const uint32_t par = static_cast<uint32_t>(it & 1);
                const int nb0 = (item % P.out_groups) * P.blocks_per_group;
                const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
                // first product
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
                        umma_f16(tmem_base, fused_operand_desc<false>(sx, ks),
                                 fused_operand_desc<BWD>(sx + C::IN_BYTES, ks), idesc_1, (kb > 0 || ks > 0) ? 1u : 0u);
                    issued_any = true;
                    umma_commit(&empty_bar[stage]);
                    next();
                }
                if (!ok) break;
                umma_commit(zfull);
                // second product, once the epilogue has written the intermediate
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
                    const uint32_t d_y = tmem_base + static_cast<uint32_t>(C::OUT_COL0 + b * FBN);
                    for (int k2 = 0; k2 < KH; ++k2) {
                        if (!wait_bounded(&full_bar[stage], phase, wc, ST_TIMEOUT_MMA)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t sb = smem_u32(ring + stage * C::STAGE_BYTES);
                        const uint32_t sh = t_addr + k2 * (BM * BK * 2);
#pragma unroll
                        for (int ks = 0; ks < BK / UMMA_K; ++ks)
                            umma_f16(d_y, fused_operand_desc<false>(sh, ks), fused_operand_desc<BWD>(sb, ks), idesc_2,
                                     (k2 > 0 || ks > 0) ? 1u : 0u);
                        umma_commit(&empty_bar[stage]);
                        next();
                    }
                    if (!ok) break;
                    umma_commit(&yfull[b]);
                }
                if (!ok) break;
                umma_commit(hempty);   // the intermediate may be overwritten once these MMAs are done
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
        const uint32_t t_addr = smem_u32(tbuf);
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
        for (int item = blockIdx.x; item < items; item += gridDim.x, ++it) {
            const uint32_t par = static_cast<uint32_t>(it & 1);
            const int row0 = (item / P.out_groups) * BM + q * 32;  // first row of this warp's 32
            const bool first = item % P.out_groups == 0;           // the item that stores the rank-r results
            const int nb0 = (item % P.out_groups) * P.blocks_per_group;
            const int nb1 = min(nb0 + P.blocks_per_group, P.n_blocks);
            // ---- the rank-r step: the intermediate into shared memory, the saved results to global memory
            if (!wait_bounded(zfull, par, wc, ST_TIMEOUT_EPILOGUE)) break;
            if (BWD) {
                if (!wait_bounded(zld, par, wc, ST_TIMEOUT_EPILOGUE)) break;
            } else {
                if (!wait_bounded(hempty, par ^ 1u, wc, ST_TIMEOUT_EPILOGUE)) break;
            }
            tc_fence_after();
            for (int c = half; c < R / 32; c += 2) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + c * 32, v);
                // row `row_in`, columns c*32 .. c*32+31 of the tile buffer: k-block c / 2, 16-byte
                // chunks 4 (c & 1) .. +3 of the 128-byte row, swizzled by the row's place in its 8-row group
                const uint32_t rbase = t_addr + (c >> 1) * (BM * BK * 2) + row_in * 128;
                uint32_t w[16];
                if (BWD) {
                    uint32_t z[16];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const uint4 t = ld_shared_v4(rbase + (((4 * (c & 1) + j) ^ (row_in & 7)) << 4));
                        z[4 * j] = t.x;
                        z[4 * j + 1] = t.y;
                        z[4 * j + 2] = t.z;
                        z[4 * j + 3] = t.w;
                    }
                    tmem_ld_wait();
                    // dZ = bf16(acc * sigma'(Z)), as the B1 epilogue of the two-GEMM backward;
                    // under CoLA-M also H = sigma(Z), from the same logistic
                    uint32_t h[16];
                    const bool want_h = P.store_s2 && first;
                    with_sigma_fixed<SIG>([&](auto tag) {
                        constexpr int S = decltype(tag)::value;
                        if constexpr (S == SIG_SILU) {
                            if (below_tanh_floor(z)) {
                                if (want_h)
                                    dsilu_silu_chunk_fallback(z, v, w, h);
                                else
                                    dsilu_chunk_fallback(z, v, w);
                                return;
                            }
                        }
                        if (want_h) {
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                float hl, dl, hh, dh;
                                act_both<S, LOGI_TANH>(bf16_lo(z[j]), hl, dl);
                                act_both<S, LOGI_TANH>(bf16_hi(z[j]), hh, dh);
                                w[j] = pack_bf16x2(__uint_as_float(v[2 * j]) * dl, __uint_as_float(v[2 * j + 1]) * dh);
                                h[j] = pack_bf16x2(hl, hh);
                            }
                        } else {
#pragma unroll
                            for (int j = 0; j < 16; ++j)
                                w[j] = pack_bf16x2(__uint_as_float(v[2 * j]) * act_dsigma<S, LOGI_TANH>(bf16_lo(z[j])),
                                                   __uint_as_float(v[2 * j + 1]) * act_dsigma<S, LOGI_TANH>(bf16_hi(z[j])));
                        }
                    });
                    if (P.store_s1 && first) emit(&P.map_s1, w, c * 32, row0);
                    if (want_h) emit(&P.map_s2, h, c * 32, row0);   // for the weight gradient of B
                } else {
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    if (P.store_s1 && first) emit(&P.map_s1, w, c * 32, row0);
                    with_sigma_fixed<SIG>([&](auto tag) {
                        constexpr int S = decltype(tag)::value;
                        if constexpr (S == SIG_SILU) {
                            if (below_tanh_floor(w)) {
                                silu_chunk_fallback(w);
                                return;
                            }
                        }
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            w[j] = pack_bf16x2(act_sigma<S, LOGI_TANH>(bf16_lo(w[j])),
                                               act_sigma<S, LOGI_TANH>(bf16_hi(w[j])));
                    });
                    if (P.store_s2 && first) emit(&P.map_s2, w, c * 32, row0);
                }
                // the intermediate (H / dZ) over the same 16-byte chunks
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    st_shared_v4(rbase + (((4 * (c & 1) + j) ^ (row_in & 7)) << 4), w[4 * j], w[4 * j + 1],
                                 w[4 * j + 2], w[4 * j + 3]);
            }
            tc_fence_before();
            mbar_arrive(zempty);                // first product read: the next tile's may start
            fence_proxy_async_smem();           // the intermediate visible to the tensor cores
            mbar_arrive(hfull);
            // ---- output blocks
            bool ok = true;
            for (int nb = nb0; nb < nb1; ++nb, ++yblk) {
                const int b = static_cast<int>(yblk & 1);
                if (!wait_bounded(&yfull[b], static_cast<uint32_t>((yblk >> 1) & 1), wc, ST_TIMEOUT_EPILOGUE)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int left = P.n_out - nb * FBN;
                const int nch = row0 >= P.n ? 0 : (left >= FBN ? FBN / 32 : (left + 31) / 32);
                for (int c = half; c < nch; c += 2) {
                    const int col0 = nb * FBN + c * 32;
                    uint32_t v[32];
                    tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                           static_cast<uint32_t>(C::OUT_COL0 + b * FBN + c * 32), v);
                    tmem_ld_wait();
                    uint32_t w[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    if ((P.n_out & 7) != 0 && col0 + 32 > P.n_out) {
                        // ragged right edge: masked per-element stores, padding untouched
                        const int row = row0 + lane;
                        if (row < P.n) {
                            uint16_t* d = reinterpret_cast<uint16_t*>(P.out_ptr + row * P.out_ld + col0);
                            const int valid = P.n_out - col0;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (j < valid) d[j] = static_cast<uint16_t>((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xFFFFu));
                        }
                        continue;
                    }
                    emit(&P.map_out, w, col0, row0);
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
