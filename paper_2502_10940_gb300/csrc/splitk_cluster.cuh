// splitk_cluster.cuh -- weight gradients whose token splits are reduced
// inside a thread-block cluster (sm_103a), for launches with few output tiles
// (a few thousand tokens):
//
//   D[tile] = sum over s = 0..S-1 of  sum over tokens t of split s of  P[t, m] Q[t, n]
//
// (dB = dY^T H, dA = dZ^T X, Sec. 3.4; P and Q token-major, read MN-major.)
//
// Each 128 x 128 output tile runs on one cluster of S CTAs (1 <= S <= 8),
// CTA s accumulating the k-blocks of split s in its own TMEM.  The partial
// tile is then reduced on chip instead of going through fp32 slabs in global
// memory and a second launch: the rows of the tile are dealt out in S bands
// of ceil(128 / S) rows (the last one shorter), CTA p owning band p.  Every CTA stages its fp32 partial in
// its own (now idle) operand ring and sends each owner that owner's band with
// one bulk copy into the owner's shared memory (cp.async.bulk
// shared::cta -> shared::cluster, counted as transaction bytes on the
// owner's mbarrier), into a slot of its own, so no two writers share an
// address.  Each owner waits for its band from all S CTAs, adds the S
// partials in the fixed order s = 0, 1, ..., S - 1 -- so every run adds the
// same numbers in the same order -- applies the epilogue and stores its rows
// with coalesced global stores.  A staged row keeps 16-byte chunk j at
// (j xor (row mod 8)): the writes of 32 rows are free of bank conflicts, and
// the owner reads the rows back in order.
//
// Epilogues (CredOp): a bf16 store, or an fp32 accumulate (D += sum, for
// gradients accumulated in fp32).  The forward GEMMs of a handful of tokens
// were run this way too, and measured no faster than their slab split with
// a reduce launch (which overlaps the GEMM's tail): 1B-shaped 32-token
// forward 0.0659 against 0.0661 ms, 7B-shaped 0.093 against 0.091 ms.
//
// The receive buffer (S bands of up to ceil(128 / S) rows, at most 133 rows
// of 128 fp32) has shared memory of its own,
// beside a 4-stage operand ring (the splits of these launches are a few
// k-blocks long), and each CTA arms its `data` barrier for the bytes it will
// receive before the cluster's start-up barrier: a CTA sends its bands as
// soon as its partial is complete, with no handshake.  (Reusing the ring for
// the receive buffer needed a "ring free" exchange among the CTAs, measured
// at 2.4-4.5 us of a 10 us launch; pushing the rows with 16-byte st.async
// stores took about 3 us per CTA.)  A CTA's staged partial must outlive the
// copies that read it: an owner whose band is complete tells every CTA so
// (an arrive on its `done` barrier), and a CTA exits only once all S have.
// All waits are bounded, as in gemm.cuh; a CTA whose own wait ran out still
// sends its bands (zeros where its accumulator is unusable), so that no other
// CTA of the cluster waits for rows that never come, and the exchange's own
// waits outlast the main loop's (4 s for the bands, 6 s for the exit signal,
// against 2 s), so that the bands of a CTA that gave up still land before
// anyone exits.
//
// Warp roles as in gemm.cuh (320 threads, one CTA per SM): warp 0 TMA
// producer, warp 1 MMA issuer (allocates TMEM), warps 2..9 the exchange and
// the reduction.
#pragma once
#include "gemm.cuh"

namespace cola {

// Copy `bytes` (a multiple of 16) from this CTA's shared memory at `src` to
// the shared memory of a CTA of this cluster at shared::cluster address
// `dst`, counted as transaction bytes on that CTA's mbarrier at
// shared::cluster address `mbar` (the copy engine, one instruction).
__device__ __forceinline__ void bulk_copy_to_cluster(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t mbar)
{
    asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     dst),
                 "r"(src), "r"(bytes), "r"(mbar)
                 : "memory");
}

// Arrive on an mbarrier of a CTA of this cluster, with no ordering of this
// thread's memory operations (a pure signal).
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t cluster_addr)
{
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// A wait of the exchange between the CTAs of a cluster.  It does not return
// early on this CTA's abort flag, since copies of other CTAs may still be on
// their way into this CTA's shared memory; its bound (`limit` ns) exceeds
// the bounds of every earlier phase of the other CTAs, so that a CTA that
// gave up on its own main loop (after WAIT_LIMIT_NS) still delivers its
// bands and signals before its peers stop waiting for them.  On expiry it
// records ST_TIMEOUT_DRAIN and returns false.
__device__ __forceinline__ bool exchange_wait(uint64_t* bar, uint64_t limit, unsigned int* status)
{
    if (mbar_try_wait_cluster(bar, 0)) return true;
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait_cluster(bar, 0)) {
        if (global_timer_ns() - t0 > limit) {
            if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
            return false;
        }
    }
    return true;
}

// Named barrier of the eight exchange warps.
__device__ __forceinline__ void exchange_warps_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

enum CredOp : int { CRED_STORE = 0, CRED_ACC = 1 };

constexpr int CBN = 128;        // tile width
constexpr int MAX_CLUSTER = 8;  // portable cluster size

struct CredProblem {
    CUtensorMap map_a, map_b;
    int M, N, k_blocks;
    int m_tiles, n_tiles;
    int tile_begin;   // first batch-wide tile of this problem
    void* out;        // CRED_STORE: bf16 D; CRED_ACC: fp32 D
    long long ldo;    // row pitch of out, elements
};

// Up to MAX_GROUP GEMMs with the same K, their tiles numbered problem after
// problem (row-major within one); tile t runs on the CTAs
// [t * S, (t + 1) * S), which form one cluster.
struct CredBatch {
    CredProblem prob[MAX_GROUP];
    int count;
    int tiles;
    int S;      // CTAs per cluster = K splits, 1 ... MAX_CLUSTER
    int kps;    // k-blocks per split (the last split may have fewer, or none)
    int op;     // CredOp
    unsigned int* status;
    // failure-detection self-test: 1 = CTA rank 1 of the first cluster issues
    // no loads, so its MMA issuer's first wait runs out while the other CTAs
    // of the cluster complete normally
    int selftest;
};

struct CredCfg {
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = CBN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGES = 4;
    static constexpr int RECV_ROWS = 136;             // >= S * ceil(128 / S) for S <= 8 (133 at S = 7)
    static constexpr int RECV_BYTES = RECV_ROWS * CBN * 4;
    static constexpr int BAR_BYTES = 256;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + RECV_BYTES + BAR_BYTES;
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static constexpr int TMEM_COLS = 128;
};

// The kernel itself is compiled in one translation unit (gemm_cluster.cu);
// the others see the batch description only.
#ifdef COLA_DEFINE_CLUSTER_KERNEL
__global__ void __launch_bounds__(NUM_THREADS, 1) splitk_cluster_kernel(const __grid_constant__ CredBatch b)
{
    using C = CredCfg;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* smem_a = smem;                            // STAGES x A_BYTES
    uint8_t* smem_b = smem + STAGES * C::A_BYTES;      // STAGES x B_BYTES
    uint8_t* recv_gen = smem + STAGES * C::STAGE_BYTES;   // [S][rows][CBN] fp32: this CTA's band from every CTA
    const uint32_t recv = smem_u32(recv_gen);
    uint64_t* bars = reinterpret_cast<uint64_t*>(recv_gen + C::RECV_BYTES);
    uint64_t* full_bar = bars;                 // [STAGES]
    uint64_t* empty_bar = bars + STAGES;       // [STAGES]
    uint64_t* tfull = bars + 2 * STAGES;       // the partial accumulated (MMA commit)
    uint64_t* data = tfull + 1;                // this CTA's band has arrived from every CTA
    uint64_t* done = data + 1;                 // every owner has received this CTA's bands (S arrivals)
    uint64_t* drain_bar = done + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    unsigned int* const status = b.status;
    const WaitCtx wc{abort_flag, status};
    const int S = b.S;
    const int RP = (BM + S - 1) / S;           // rows of a band; band p: rows [p RP, p RP + band_rows(p))
    const uint32_t rank = cluster_ctarank();
    auto band_rows = [&](int p) { return min(RP, BM - p * RP); };
    const int my_rows = band_rows(static_cast<int>(rank));
    const int tile = static_cast<int>(blockIdx.x) / S;
    int g = 0;
#pragma unroll
    for (int j = 1; j < MAX_GROUP; ++j)
        if (j < b.count && tile >= b.prob[j].tile_begin) g = j;
    const CredProblem& P = b.prob[g];
    const int t = tile - P.tile_begin;
    const int m_blk = t / P.n_tiles, n_blk = t - (t / P.n_tiles) * P.n_tiles;
    const int kb0 = static_cast<int>(rank) * b.kps;
    const int kb1 = min(kb0 + b.kps, P.k_blocks);
    const bool has_k = kb0 < kb1;              // a split past the end of K adds zeros

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        mbar_init(tfull, 1);
        mbar_init(data, 1);
        mbar_init(done, static_cast<uint32_t>(S));
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_mbar_init();
        // armed before any CTA of the cluster can send: my band from each of the S CTAs
        mbar_arrive_expect_tx(data, static_cast<uint32_t>(S * my_rows * CBN * 4));
        tma_prefetch_desc(&P.map_a);
        tma_prefetch_desc(&P.map_b);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    cluster_sync();   // every CTA's barriers initialised before any arrives from another
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
            const int m0 = m_blk * BM, n0 = n_blk * CBN;
            const bool no_loads = b.selftest == 1 && tile == 0 && rank == 1;
            for (int kb = kb0; kb < kb1 && !no_loads; ++kb) {
                if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                    ok = false;
                    break;
                }
                uint8_t* sa = smem_a + stage * C::A_BYTES;
                uint8_t* sb = smem_b + stage * C::B_BYTES;
                mbar_arrive_expect_tx(&full_bar[stage], C::STAGE_BYTES);
                // MN-major operands: 64-column boxes along M (N), 64 tokens deep
#pragma unroll
                for (int j = 0; j < BM / 64; ++j) tma_load_2d(&P.map_a, &full_bar[stage], sa + j * 64 * BK * 2, m0 + 64 * j, kb * BK);
#pragma unroll
                for (int j = 0; j < CBN / 64; ++j) tma_load_2d(&P.map_b, &full_bar[stage], sb + j * 64 * BK * 2, n0 + 64 * j, kb * BK);
                ++issued;
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
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
                            if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                            break;
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(BM, CBN, 1, 1);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true, issued_any = false;
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
                    // next 16 tokens: +16 rows of 128 bytes; 64-column groups 8 KB apart
                    const uint64_t da = smem_desc_sw128(sa + ks * UMMA_K * 128, 64 * BK * 2, 1024);
                    const uint64_t db = smem_desc_sw128(sb + ks * UMMA_K * 128, 64 * BK * 2, 1024);
                    umma_f16(tmem_base, da, db, idesc, (kb > kb0 || ks > 0) ? 1u : 0u);
                }
                issued_any = true;
                umma_commit(&empty_bar[stage]);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            // the partial is complete (with no k-block, at once: nothing in flight)
            umma_commit(tfull);
            if ((!ok || *abort_flag) && issued_any) {
                umma_commit(drain_bar);
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0)) {
                    if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                        if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------ exchange and reduction (warps 2..9)
        const int q = warp & 3;                 // TMEM lane quarter
        const int half = (warp - 2) >> 2;       // alternate 32-column chunks
        const int row = q * 32 + lane;          // this thread's row of the partial tile
        const bool acc_ok = wait_bounded(tfull, 0, wc, ST_TIMEOUT_EPILOGUE);
        tc_fence_after();
        // stage this row's partial in the ring: row-major fp32, 16-byte chunk j
        // of the row at (j xor (row mod 8))
        const uint32_t stg = smem_u32(smem) + static_cast<uint32_t>(row * CBN * 4);
        // an accumulator this CTA gave up on sends zeros (tcgen05.ld is warp-wide)
        const bool use_acc = __all_sync(0xffffffffu, acc_ok && has_k && !*abort_flag);
#pragma unroll
        for (int i = 0; i < CBN / 64; ++i) {
            const int c = half + 2 * i;
            uint32_t v[32];
            if (use_acc) {
                tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(c * 32), v);
                tmem_ld_wait();
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = 0u;
            }
#pragma unroll
            for (int j = 0; j < 8; ++j)
                st_shared_v4(stg + static_cast<uint32_t>(((c * 8 + j) ^ (row & 7)) << 4), v[4 * j], v[4 * j + 1],
                             v[4 * j + 2], v[4 * j + 3]);
        }
        tc_fence_before();
        fence_proxy_async_smem();   // the staged rows visible to the copy engine
        exchange_warps_sync();
        const int tid = threadIdx.x - 64;
        if (tid < S) {
            // band `tid` of this partial into slot `rank` of its owner (slots of band_rows(tid) rows)
            const uint32_t bytes = static_cast<uint32_t>(band_rows(tid) * CBN * 4);
            bulk_copy_to_cluster(mapa_shared(recv + rank * bytes, static_cast<uint32_t>(tid)),
                                 smem_u32(smem) + static_cast<uint32_t>(tid * RP * CBN * 4), bytes,
                                 mapa_shared(smem_u32(data), static_cast<uint32_t>(tid)));
        }
        // this CTA's band from every CTA, summed in CTA order
        const bool dok = exchange_wait(data, 2 * WAIT_LIMIT_NS, status);
        // every copy into this CTA has landed: tell each sender that its band
        // here has been read
        if (tid < S) mbar_arrive_cluster_relaxed(mapa_shared(smem_u32(done), static_cast<uint32_t>(tid)));
        if (dok && !*abort_flag) {
            const int items = my_rows * (CBN / 4);
            for (int it = tid; it < items; it += NUM_EPI_WARPS * 32) {
                const int lr = it / (CBN / 4), c4 = it - lr * (CBN / 4);
                // slot s, row lr: row rank * RP + lr of every sender's staging
                const int pos = (c4 ^ ((static_cast<int>(rank) * RP + lr) & 7)) * 4;
                float4 a = *reinterpret_cast<const float4*>(recv_gen + (lr * CBN + pos) * 4);
                for (int s = 1; s < S; ++s) {
                    const float4 u = *reinterpret_cast<const float4*>(recv_gen + ((s * my_rows + lr) * CBN + pos) * 4);
                    a.x += u.x;
                    a.y += u.y;
                    a.z += u.z;
                    a.w += u.w;
                }
                const int gr = m_blk * BM + static_cast<int>(rank) * RP + lr;
                const int gc = n_blk * CBN + c4 * 4;
                if (gr >= P.M || gc >= P.N) continue;
                const int valid = min(4, P.N - gc);
                const float v[4] = {a.x, a.y, a.z, a.w};
                const long long off = static_cast<long long>(gr) * P.ldo + gc;
                if (b.op == CRED_ACC) {
                    float* o = static_cast<float*>(P.out) + off;
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (e < valid) o[e] += v[e];
                } else {
                    const uint32_t w0 = pack_bf16x2(v[0], v[1]), w1 = pack_bf16x2(v[2], v[3]);
                    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(P.out) + off;
                    if (valid == 4 && (reinterpret_cast<uintptr_t>(o) & 7) == 0) {
                        *reinterpret_cast<uint2*>(o) = make_uint2(w0, w1);
                    } else {
                        uint16_t* o16 = reinterpret_cast<uint16_t*>(o);
                        const uint32_t w[2] = {w0, w1};
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (e < valid) o16[e] = static_cast<uint16_t>((e & 1) ? (w[e >> 1] >> 16) : (w[e >> 1] & 0xFFFFu));
                    }
                }
            }
        }
        // the bands this CTA sent have been read by their owners: its staging
        // may go away with it
        if (threadIdx.x == 64) exchange_wait(done, 3 * WAIT_LIMIT_NS, status);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}
#endif  // COLA_DEFINE_CLUSTER_KERNEL

}  // namespace cola
