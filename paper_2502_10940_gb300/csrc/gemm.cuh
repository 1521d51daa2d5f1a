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
// CTA pairs (PAIR = true): two CTAs of a cluster run one 256-row tile with
// tcgen05 cta_group::2.  Each CTA loads its own 128 rows of A and half of the
// tile's B columns; the even CTA issues M = 256 MMAs that read both CTAs'
// shared memory and accumulate each CTA's 128 rows in that CTA's TMEM.  The
// per-CTA B traffic (TMA fills and MMA operand reads) halves, which relieves
// the shared-memory bandwidth that bounds a single-CTA M = 128 GEMM.  Both
// CTAs' TMA loads count on the even CTA's stage barrier; its MMA commits
// arrive on the stage and accumulator barriers of both CTAs; the odd CTA's
// epilogue arrives on the even CTA's accumulator-free barrier.
//
// Warp roles (320 threads, one CTA per SM, persistent over output tiles):
//   warp 0      TMA producer: fills a STAGES-deep ring of (A, B) k-blocks.
//   warp 1      MMA issuer:  tcgen05.mma M=128 (M=256 on a CTA pair, issued
//               by its even CTA), N=BN, K=16 into one of two TMEM
//               accumulators (double buffered, so the epilogue of tile i
//               overlaps the main loop of tile i+1); allocates TMEM.
//   warps 2..9  epilogue, two warps per TMEM lane quarter taking alternate
//               32-column chunks: tcgen05.ld -> fused elementwise -> 32x32
//               boxes staged in shared memory (64-byte swizzle, bank-conflict
//               free) -> TMA bulk tensor stores, which are coalesced,
//               asynchronous and clipped to the tensor's extents in hardware.
//
// Epilogues (the elementwise parts of the layer, fused so that the rank-r
// intermediate makes no extra HBM round trip):
//   EPI_STORE   D = bf16(acc)                                  (Y, dX)
//   EPI_ZH      Z = bf16(acc), H = bf16(sigma(Z))              (forward A-GEMM)
//   EPI_DSIGMA  dZ = bf16(acc * sigma'(Z_saved)); EPI_DSIGMA_H (CoLA-M) also
//               H = bf16(sigma(Z_saved)) for the weight gradient of B
//   EPI_F32     fp32 split-K partial slab, reduced (in a fixed order) by the
//               reduce kernel: fp32-accumulated weight gradients, and the
//               forward GEMMs of small launches
//   EPI_GLU     gated MLP forward (Fig. 4): the K walk covers [H_gate H_up]
//               (2r columns of H_cat); the gate half accumulates H_gate B_gate^T
//               and the up half H_up B_up^T into a second accumulator of the
//               same tile, and the epilogue stores M = bf16(Y_gate * Y_up) of
//               the bf16-rounded outputs (and Y_gate, Y_up when training)
//   EPI_GLU_BWD dX GEMM of the down layer whose input is that M: with
//               dM = bf16(acc) it stores dY_gate = bf16(dM * Y_up) and
//               dY_up = bf16(dM * Y_gate), reading Y_gate, Y_up per chunk
//   EPI_TAIL      weight gradients (bf16 D) with a split tail: the tiles of
//               the full waves run whole and store D = bf16(acc) as
//               EPI_STORE; the tiles of the last, partial wave are split
//               over K into pieces that store fp32 partials into slots, which
//               the tail reduce sums in a fixed order
//
// Every mbarrier wait is bounded (WAIT_LIMIT_NS of global time).  On expiry
// the waiting thread records where it gave up in the status word, raises a
// CTA-wide abort flag that makes every other wait return, waits (bounded) for
// its own copies and MMAs still in flight, and the CTA frees its TMEM and
// exits.  No wait can spin forever.
//
// On a CTA pair the odd CTA's TMA loads complete on the even CTA's stage
// barriers, so it cannot see them land itself.  At the end of the producer
// role the odd producer reports how many k-blocks it issued (a store into
// the even CTA's shared memory, published by a cluster-scope release arrive
// on the even CTA's exchange barrier) and waits for the even CTA's relay.
// The even producer, after an abort, reconciles the stage phases that the two
// producers left unequal -- it arms the phases only the odd CTA issued (for
// the odd CTA's bytes) and completes the odd CTA's share of the phases only
// it issued -- waits for every phase still outstanding, so that every load of
// either CTA has landed, and then arrives on the odd CTA's relay barrier.
#pragma once
#include <cuda_bf16.h>
#include <cstdint>

#include "ptx.cuh"

namespace cola {

constexpr int BM = 128;              // UMMA M (cta_group::1): one row per TMEM lane
constexpr int BK = 64;               // k-block: one 128-byte swizzle row of bf16
constexpr int UMMA_K = 16;           // K of one kind::f16 MMA
constexpr int NUM_EPI_WARPS = 8;     // two per TMEM lane quarter
constexpr int NUM_THREADS = 64 + 32 * NUM_EPI_WARPS;
constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;   // 2 s

// bits recorded in the status word when a wait gives up
enum : unsigned int {
    ST_TIMEOUT_PRODUCER = 1u << 0,
    ST_TIMEOUT_MMA = 1u << 1,
    ST_TIMEOUT_EPILOGUE = 1u << 2,
    ST_TIMEOUT_DRAIN = 1u << 3,
};

enum Epi : int {
    EPI_STORE = 0, EPI_ZH = 1, EPI_DSIGMA = 2, EPI_F32 = 3, EPI_TAIL = 4, EPI_GLU = 5, EPI_GLU_BWD = 6,
    EPI_DSIGMA_H = 7
};
enum Sigma : int { SIG_IDENTITY = 0, SIG_SILU = 1, SIG_GELU = 2 };

struct GemmParams {
    int M, N;              // logical output extents
    int k_blocks;          // ceil(K / BK)
    int m_tiles, n_tiles;
    int splits, kb_per_split;
    int units;             // m_tiles * n_tiles * splits
    void* D;               // EPI_F32: fp32 partial slabs (bf16 outputs go through map_d / map_d2)
    long long ldd;         // EPI_F32: row pitch of a slab in elements
    long long part_stride; // EPI_F32: elements per split slab
    int has_d2;            // EPI_ZH: also store H through map_d2 (EPI_DSIGMA_H always does)
    int h_only;            // EPI_ZH: store H = sigma(bf16(acc)) through map_d and nothing else
    // tile order within the problem: 0 = row-major (n_blk fastest), 1 =
    // column-major (m_blk fastest).  A wave of CTAs walking the reduction in
    // step reads each B-operand panel of its tiles once; column-major keeps a
    // wave on few B panels, for problems whose B operand is the larger one.
    int n_major;
    // The bf16 output behind map_d, for the one 32-column chunk per row block
    // that holds a ragged right edge (N % 8 != 0): a TMA store clips at
    // 16-byte granularity and would write the row padding past column N, so
    // that chunk is stored with masked direct stores instead.
    __nv_bfloat16* d_ptr;
    long long d_ld;
    int sigma;
    unsigned int* status;
    // gated MLP (EPI_GLU, EPI_GLU_BWD): the outputs behind map_d2 and map_d3,
    // for the masked stores of a ragged right edge (pitch d_ld), and the
    // Y_gate, Y_up that the EPI_GLU_BWD epilogue reads (pitch d_ld)
    int glu_half;                 // EPI_GLU: k-blocks of the gate half; the up half reads map_b2
    __nv_bfloat16* d2_ptr;
    __nv_bfloat16* d3_ptr;
    const __nv_bfloat16* yg_ptr;
    const __nv_bfloat16* yu_ptr;
    // problem 0 only, for the failure-detection self-tests: 1 = the producers
    // issue nothing, so the MMA's first wait runs out; 2 = the odd CTA of a
    // pair issues its first k-block only, so the MMA's second wait runs out
    // with the even CTA's loads of later stages in flight or landed
    int selftest;
};

// Epilogue staging: per epilogue warp two 2 KB boxes of 32 rows x 32 bf16
// columns (64-byte rows, 64-byte TMA swizzle).  EPI_STORE / EPI_ZH / EPI_GLU /
// EPI_GLU_BWD use them as a ring of output boxes.  EPI_DSIGMA uses them as a double buffer for the
// saved Z: the box of the warp's next chunk is TMA-loaded while the current
// one is processed, and dZ is computed in place and TMA-stored from the box.
constexpr int EPI_BOX_BYTES = 32 * 32 * 2;
constexpr int EPI_OUT_BOXES = 2;
static_assert(EPI_OUT_BOXES == 2, "the CTA-pair store epilogue stages a chunk pair into the whole ring");
constexpr int EPI_WARP_BYTES = EPI_OUT_BOXES * EPI_BOX_BYTES;
constexpr int EPI_SMEM_BYTES = NUM_EPI_WARPS * EPI_WARP_BYTES;

// A CTA tile is MSUB x 128 rows by BN columns: MSUB = 2 runs two M = 128
// MMAs per k-step that share one B tile (halving the B-operand traffic per
// output row), into two TMEM accumulators of BN columns each.  ACCS = 2: one
// 128-row tile with two accumulators (the gate and up halves of EPI_GLU).
// BUFS: tiles whose accumulators TMEM holds at once (2: the epilogue of one
// tile overlaps the main loop of the next).
template <int BN, int MSUB, bool PAIR = false, int ACCS = 1, int BUFS = 2>
struct GemmCfg {
    static_assert(BN % 64 == 0 && BN >= 64 && BN <= 256, "BN must be 64..256 in steps of 64");
    static_assert(MSUB == 1 || MSUB == 2, "one or two 128-row sub-tiles");
    static_assert(!PAIR || (MSUB == 1 && BN >= 128), "a CTA pair runs 128 rows and BN / 2 >= 64 B columns per CTA");
    static constexpr int TILE_M = PAIR ? 2 * BM : BM * MSUB;   // rows of one unit
    static constexpr int CTA_ROWS = PAIR ? BM : TILE_M;          // rows of A this CTA loads
    static constexpr int B_ROWS = PAIR ? BN / 2 : BN;           // columns of B this CTA loads
    static constexpr int ACC_COLS = (MSUB > ACCS ? MSUB : ACCS) * BN;   // TMEM columns of one tile's accumulators
    static_assert(BUFS * ACC_COLS <= 512, "the accumulators must fit TMEM");
    static constexpr int A_BYTES = CTA_ROWS * BK * 2;
    static constexpr int B_BYTES = B_ROWS * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int BAR_BYTES = 512;        // 39 mbarriers, the TMEM address, the abort flag, a count
    static constexpr int SMEM_LIMIT = 232448;   // opt-in maximum per CTA
    static constexpr int STAGES_FIT = (SMEM_LIMIT - 1024 - BAR_BYTES - EPI_SMEM_BYTES) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
    static constexpr int TMEM_COLS = (BUFS * ACC_COLS <= 128) ? 128 : (BUFS * ACC_COLS <= 256 ? 256 : 512);
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + EPI_SMEM_BYTES + BAR_BYTES;
    static_assert(SMEM_BYTES <= SMEM_LIMIT, "shared memory budget");
};

// two bf16 values packed in a 32-bit word (low half first) and back
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// ------------------------------------------------------------ activations
// The logistic s(z) = 1 / (1 + e^{-z}) of SiLU, in two forms:
//   tanh form         s = 1/2 + tanh(z/2)/2 with tanh from the special-function
//   (logistic_tanh)   unit's approximation: one MUFU operation per element.
//                     For z < 0 the sum cancels (s -> 0 while tanh -> -1), so
//                     this form serves only z >= -TANH_FLOOR, where its
//                     relative error stays below 1e-4 (measured on every bf16
//                     input: a twentieth of half a bf16 ulp).
//   exponential form  s = 1 / (1 + e^{-z}) with the fast exponential and
//   (logistic_exp)    divide (a few ulp of fp32): two MUFU operations; exactly
//                     0 below -87, where e^{-z} would leave the range of the
//                     fast divide.
// The value of every element is logistic_of<LOGI_SELECT>(z): the exponential
// form below -TANH_FLOOR, the tanh form elsewhere.  The epilogues evaluate a
// chunk of a row (32 values) with no input below the floor (under N(0, 1)
// inputs, all but about 3 chunks in 10^8) by the tanh form alone
// (logistic_of<LOGI_TANH>), and any other chunk element by element with the
// choice, out of line (the *_chunk_select functions below), so a result never
// depends on its neighbours.  The SFU rate bounds the sigma epilogues of the
// HBM-bound launches, which the single-operation form relieves.  Every sigma
// input is a bf16 value (the stored Z); over all of them the result is
// checked through the library against the oracle.
constexpr float TANH_FLOOR = 6.0f;
constexpr uint32_t TANH_FLOOR_BF16_NEG = 0xC0C0u;   // bf16 bit pattern of -6.0
enum { LOGI_TANH = 0, LOGI_SELECT = 1 };

__device__ __forceinline__ float logistic_tanh(float z)
{
    float t;
    asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(0.5f * z));
    return fmaf(0.5f, t, 0.5f);
}

__device__ __forceinline__ float logistic_exp(float z)
{
    return z < -87.0f ? 0.0f : __fdividef(1.0f, 1.0f + __expf(-z));
}

template <int L>
__device__ __forceinline__ float logistic_of(float z)
{
    if (L == LOGI_TANH) return logistic_tanh(z);
    return z < -TANH_FLOOR ? logistic_exp(z) : logistic_tanh(z);
}

// Whether any of the 2N bf16 values packed in w lies below -TANH_FLOOR
// (negative with a magnitude above the floor's: as unsigned 16-bit patterns,
// above -6.0's; NaN patterns with the sign bit set count too, harmlessly).
template <int N>
__device__ __forceinline__ bool below_tanh_floor(const uint32_t (&w)[N])
{
    uint32_t m = 0;
#pragma unroll
    for (int j = 0; j < N; ++j) m = __vmaxu2(m, w[j]);
    return (m & 0xFFFFu) > TANH_FLOOR_BF16_NEG || (m >> 16) > TANH_FLOOR_BF16_NEG;
}

template <int SIG, int L = LOGI_SELECT>
__device__ __forceinline__ float act_sigma(float z)
{
    if (SIG == SIG_SILU) return z * logistic_of<L>(z);
    if (SIG == SIG_GELU) return 0.5f * z * erfcf(-z * 0.70710678118654752f);
    return z;
}

template <int SIG, int L = LOGI_SELECT>
__device__ __forceinline__ float act_dsigma(float z)
{
    if (SIG == SIG_SILU) {
        const float s = logistic_of<L>(z);
        return s * (1.0f + z * (1.0f - s));
    }
    if (SIG == SIG_GELU) {
        const float Phi = 0.5f * erfcf(-z * 0.70710678118654752f);
        const float phi = 0.39894228040143268f * __expf(-0.5f * z * z);
        return Phi + z * phi;
    }
    return 1.0f;
}

// sigma(z) and sigma'(z) together, sharing the logistic (SiLU) or the normal
// CDF and density (GELU): the same values as act_sigma and act_dsigma.
template <int SIG, int L = LOGI_SELECT>
__device__ __forceinline__ void act_both(float z, float& h, float& d)
{
    if (SIG == SIG_SILU) {
        const float s = logistic_of<L>(z);
        h = z * s;
        d = s * (1.0f + z * (1.0f - s));
    } else if (SIG == SIG_GELU) {
        const float Phi = 0.5f * erfcf(-z * 0.70710678118654752f);
        const float phi = 0.39894228040143268f * __expf(-0.5f * z * z);
        h = z * Phi;   // = (0.5 z) erfc(...) of act_sigma: scaling by 0.5 is exact
        d = Phi + z * phi;
    } else {
        h = z;
        d = 1.0f;
    }
}

template <int SIG>
struct SigTag {
    static constexpr int value = SIG;
};

// Run fn(SigTag<SIG>{}): the activation of a kernel specialised for one
// sigma, so the unrolled elementwise loops carry no branch on the activation
// kind.  Every kernel whose epilogue evaluates sigma is compiled once per
// activation: a kernel then holds only its own activation's code, and the
// small launches, whose code runs once per CTA from a cold instruction cache,
// fetch less of it (measured: the 2048-token layer step 12 % faster than with
// the three activations behind a run-time switch in one kernel).
template <int SIG, class Fn>
__device__ __forceinline__ void with_sigma_fixed(Fn&& fn)
{
    fn(SigTag<SIG>{});
}

// The SiLU steps of one epilogue chunk (a row's 32 values, 16 packed bf16
// pairs) that holds an input below the tanh form's floor: every element
// takes logistic_of<LOGI_SELECT>.  Out of line, so that the unrolled loops of
// the common chunk (LOGI_TANH) stay compact: measured, inlining both forms
// cost the small launches more in cold instruction fetches than the rare
// call costs here.  Arguments and results pass by value.
struct Words16 {
    uint32_t w[16];
};
struct Words32 {
    uint32_t w[32];
};

static __device__ __noinline__ Words16 silu_chunk_select(Words16 z)
{
    Words16 h;
#pragma unroll
    for (int j = 0; j < 16; ++j)
        h.w[j] = pack_bf16x2(act_sigma<SIG_SILU>(bf16_lo(z.w[j])), act_sigma<SIG_SILU>(bf16_hi(z.w[j])));
    return h;
}

// dZ = bf16(acc * sigma'(Z)) for a chunk of fp32 accumulators acc
static __device__ __noinline__ Words16 dsilu_chunk_select(Words16 z, Words32 acc)
{
    Words16 d;
#pragma unroll
    for (int j = 0; j < 16; ++j)
        d.w[j] = pack_bf16x2(__uint_as_float(acc.w[2 * j]) * act_dsigma<SIG_SILU>(bf16_lo(z.w[j])),
                             __uint_as_float(acc.w[2 * j + 1]) * act_dsigma<SIG_SILU>(bf16_hi(z.w[j])));
    return d;
}

// dZ (words 0..15) and H = sigma(Z) (words 16..31) together
static __device__ __noinline__ Words32 dsilu_silu_chunk_select(Words16 z, Words32 acc)
{
    Words32 o;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        float hl, dl, hh, dh;
        act_both<SIG_SILU>(bf16_lo(z.w[j]), hl, dl);
        act_both<SIG_SILU>(bf16_hi(z.w[j]), hh, dh);
        o.w[j] = pack_bf16x2(__uint_as_float(acc.w[2 * j]) * dl, __uint_as_float(acc.w[2 * j + 1]) * dh);
        o.w[16 + j] = pack_bf16x2(hl, hh);
    }
    return o;
}

// In-register front ends of the three: w = sigma(w); w = dZ; w = dZ, h = H.
__device__ __forceinline__ void silu_chunk_fallback(uint32_t (&w)[16])
{
    Words16 a;
#pragma unroll
    for (int j = 0; j < 16; ++j) a.w[j] = w[j];
    a = silu_chunk_select(a);
#pragma unroll
    for (int j = 0; j < 16; ++j) w[j] = a.w[j];
}

__device__ __forceinline__ void dsilu_chunk_fallback(const uint32_t (&z)[16], const uint32_t (&v)[32], uint32_t (&w)[16])
{
    Words16 a;
    Words32 b;
#pragma unroll
    for (int j = 0; j < 16; ++j) a.w[j] = z[j];
#pragma unroll
    for (int j = 0; j < 32; ++j) b.w[j] = v[j];
    a = dsilu_chunk_select(a, b);
#pragma unroll
    for (int j = 0; j < 16; ++j) w[j] = a.w[j];
}

__device__ __forceinline__ void dsilu_silu_chunk_fallback(const uint32_t (&z)[16], const uint32_t (&v)[32],
                                                          uint32_t (&w)[16], uint32_t (&h)[16])
{
    Words16 a;
    Words32 b;
#pragma unroll
    for (int j = 0; j < 16; ++j) a.w[j] = z[j];
#pragma unroll
    for (int j = 0; j < 32; ++j) b.w[j] = v[j];
    b = dsilu_silu_chunk_select(a, b);
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        w[j] = b.w[j];
        h[j] = b.w[16 + j];
    }
}

// --------------------------------------------------------- bounded waits
struct WaitCtx {
    volatile int* abort_flag;
    unsigned int* status;
};

template <bool CLUSTER = false>
__device__ __forceinline__ bool try_wait_scoped(uint64_t* bar, uint32_t parity)
{
    return CLUSTER ? mbar_try_wait_cluster(bar, parity) : mbar_try_wait(bar, parity);
}

// CLUSTER: the barrier receives arrivals from the peer CTA of a pair
// (acquire at cluster scope).
template <bool CLUSTER = false>
__device__ __forceinline__ bool wait_bounded(uint64_t* bar, uint32_t parity, const WaitCtx& w, unsigned int code)
{
    if (try_wait_scoped<CLUSTER>(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (try_wait_scoped<CLUSTER>(bar, parity)) return true;
        if (*w.abort_flag) return false;
        if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
            *w.abort_flag = 1;
            if (w.status) atomicOr(w.status, code);
            return false;
        }
    }
}

// The (m_blk, n_blk) of tile `t` of a problem in its tile order.
__host__ __device__ __forceinline__ void tile_coords(const GemmParams& p, int t, int& m_blk, int& n_blk)
{
    if (p.n_major) {
        n_blk = t / p.m_tiles;
        m_blk = t - n_blk * p.m_tiles;
    } else {
        m_blk = t / p.n_tiles;
        n_blk = t - m_blk * p.n_tiles;
    }
}

__device__ __forceinline__ void decode_unit(const GemmParams& p, int u, int& m_blk, int& n_blk, int& split,
                                            int& kb0, int& kb1)
{
    const int tiles = p.m_tiles * p.n_tiles;
    split = u / tiles;
    const int rem = u - split * tiles;
    tile_coords(p, rem, m_blk, n_blk);
    kb0 = split * p.kb_per_split;
    kb1 = min(kb0 + p.kb_per_split, p.k_blocks);
}

constexpr int MAX_GROUP = 4;

// One GEMM of a batch: its operand / output tensor maps and parameters.
struct GemmProblem {
    CUtensorMap map_a, map_b, map_d, map_d2, map_z;
    CUtensorMap map_b2, map_d3;   // EPI_GLU: B_up, and the Y_up output
    GemmParams p;
    int unit_begin;   // first batch-wide unit index of this problem
};

// Up to MAX_GROUP independent GEMMs of one configuration (tile shape,
// operand majors, epilogue) run by a single persistent launch; their work
// units are numbered consecutively, problem after problem.
//
// EPI_TAIL (split tail): the problems share K; their output tiles, problem
// after problem and row-major within one, are numbered batch-wide
// (tile_begin[g] is the first tile of problem g).  Units [0, tail_body) are
// the whole tiles 0 .. tail_body - 1 (the full waves), followed by the
// tail_tiles tiles of the last wave in tail_pieces pieces each: unit tail_body + j is
// piece j % tail_pieces of tile tail_body + j / tail_pieces, k-blocks
// [piece * tail_kps, +tail_kps) clipped to K.  With tail_pieces > 1 piece j
// stores its fp32 partial into slot j (TILE_M x BN fp32) of tail_part.
struct GemmBatch {
    GemmProblem prob[MAX_GROUP];
    int count;
    int units;
    int tail_body, tail_tiles, tail_pieces, tail_kps;
    int tile_begin[MAX_GROUP];
    float* tail_part;
};

struct Unit {
    int g, m_blk, n_blk, split, kb0, kb1;
};

__device__ __forceinline__ Unit decode(const GemmBatch& b, int u)
{
    int g = 0;
#pragma unroll
    for (int j = 1; j < MAX_GROUP; ++j)
        if (j < b.count && u >= b.prob[j].unit_begin) g = j;
    Unit x;
    x.g = g;
    decode_unit(b.prob[g].p, u - b.prob[g].unit_begin, x.m_blk, x.n_blk, x.split, x.kb0, x.kb1);
    return x;
}

// This CTA's walk over its work: units u = first_unit, first_unit + step,
// ...  The producer, MMA and epilogue roles walk the same sequence.
struct WorkIter {
    int u;   // next unit
};

template <int EPI>
__device__ __forceinline__ void work_begin(const GemmBatch&, int first_unit, WorkIter& it)
{
    it.u = first_unit;
}

// The next unit of the walk; false once the walk is over.  EPI_TAIL: a unit
// that covers its whole tile has split = -1, a piece of a split tail tile
// has split = its partial slot.
template <int EPI>
__device__ __forceinline__ bool work_next(const GemmBatch& b, int unit_step, WorkIter& it, Unit& x)
{
    if (it.u >= b.units) return false;
    const int u = it.u;
    it.u += unit_step;
    if constexpr (EPI == EPI_TAIL) {
        int t, k0 = 0, split = -1;
        int k1 = b.prob[0].p.k_blocks;
        if (u < b.tail_body) {
            t = u;
        } else {
            const int j = u - b.tail_body;
            const int piece = j % b.tail_pieces;
            t = b.tail_body + j / b.tail_pieces;
            if (b.tail_pieces > 1) {
                k0 = piece * b.tail_kps;
                k1 = min(k1, k0 + b.tail_kps);
                split = j;
            }
        }
        int g = 0;
#pragma unroll
        for (int q = 1; q < MAX_GROUP; ++q)
            if (q < b.count && t >= b.tile_begin[q]) g = q;
        x.g = g;
        tile_coords(b.prob[g].p, t - b.tile_begin[g], x.m_blk, x.n_blk);
        x.split = split;
        x.kb0 = k0;
        x.kb1 = k1;
    } else {
        x = decode(b, u);
    }
    return true;
}

// Byte offset of 16-byte chunk j of row i inside a 32 x 32 bf16 box laid out
// with the TMA 64-byte swizzle (chunk bits 4-5 XOR address bits 7-8).
__device__ __forceinline__ uint32_t box64_off(int i, int j) { return i * 64 + ((j ^ ((i >> 1) & 3)) << 4); }

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr)
{
    uint4 v;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr)
                 : "memory");
    return v;
}

// Write this thread's 32 packed bf16 (row `lane` of the box) into a staging box.
__device__ __forceinline__ void stage_row(uint32_t box, int lane, const uint32_t (&w)[16])
{
#pragma unroll
    for (int j = 0; j < 4; ++j) st_shared_v4(box + box64_off(lane, j), w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
}

// ------------------------------------------------------------ the kernel
template <int BN, int MSUB, bool A_MN, bool B_MN, int EPI, bool PAIR = false, int SIG = SIG_IDENTITY>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_kernel(const __grid_constant__ GemmBatch batch)
{
    // EPI_GLU with 256-column tiles: the gate and up accumulators of one tile
    // fill TMEM, so there is one tile slot, and its two accumulators are
    // released apart: the epilogue copies the gate half to registers and frees
    // it at once (tempty_bar[0]), so the MMAs of the next tile's gate half
    // overlap this tile's up-half epilogue; the up half is freed when stored
    // (tempty_bar[1]).
    constexpr bool GLU_SPLIT = EPI == EPI_GLU && BN == 256;
    // EPI_STORE on a CTA pair: the accumulator is freed as soon as the
    // epilogue holds the tile's values in registers, before its stores
    // (measured: the 1B Y and dX GEMMs 2-3 % faster, the 7B ones unchanged;
    // the single-CTA GEMMs of the LLaMA-60M block 5-7 % slower, which keep
    // freeing it after their stores)
    constexpr bool EARLY_FREE = EPI == EPI_STORE && PAIR;
    // the dZ epilogue: EPI_DSIGMA_H (CoLA-M) also stores H = sigma(Z), formed
    // with sigma'(Z) from one logistic; a kind of its own so that the
    // register budget of the CoLA form (dZ alone) is unaffected (measured:
    // a run-time switch between the two made the LLaMA-60M dZ GEMMs 4-10 %
    // slower)
    constexpr bool DSIG = EPI == EPI_DSIGMA || EPI == EPI_DSIGMA_H;
    using C = GemmCfg<BN, MSUB, PAIR, EPI == EPI_GLU ? 2 : 1, GLU_SPLIT ? 1 : 2>;
    constexpr int STAGES = C::STAGES;
    constexpr int TILE_M = C::TILE_M;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* smem_a = smem;                              // STAGES x A_BYTES
    uint8_t* smem_b = smem + STAGES * C::A_BYTES;        // STAGES x B_BYTES
    uint8_t* smem_epi = smem + STAGES * C::STAGE_BYTES;  // NUM_EPI_WARPS x EPI_WARP_BYTES
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem_epi + EPI_SMEM_BYTES);
    uint64_t* full_bar = bars;                 // [STAGES]
    uint64_t* empty_bar = bars + STAGES;       // [STAGES]
    uint64_t* tfull_bar = bars + 2 * STAGES;   // [2]
    uint64_t* tempty_bar = tfull_bar + 2;      // [2]
    uint64_t* drain_bar = tempty_bar + 2;      // [1]
    uint64_t* zfull_bar = drain_bar + 1;       // [NUM_EPI_WARPS][2]  Z boxes (EPI_DSIGMA)
    uint64_t* xchg_bar = zfull_bar + 2 * NUM_EPI_WARPS;   // [1] PAIR: the odd producer's report (even CTA)
    uint64_t* relay_bar = xchg_bar + 1;        // [1] PAIR: the even CTA's drain is done (odd CTA)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(relay_bar + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* odd_issued = reinterpret_cast<volatile int*>(tmem_slot + 2);   // PAIR: written by the odd CTA

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    unsigned int* const status = batch.prob[0].p.status;
    const WaitCtx wc{abort_flag, status};
    // units: one per CTA, or one per CTA pair (both CTAs of a pair take the same units)
    const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
    const bool leader = rank == 0;
    const int first_unit = PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
    const int unit_step = PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&tfull_bar[b], 1);
            mbar_init(&tempty_bar[b], NUM_EPI_WARPS * 32 * (PAIR ? 2 : 1));   // PAIR: both CTAs' epilogues
        }
        mbar_init(drain_bar, 1);
        for (int j = 0; j < 2 * NUM_EPI_WARPS; ++j) mbar_init(&zfull_bar[j], 1);
        mbar_init(xchg_bar, 1);
        mbar_init(relay_bar, 1);
        *abort_flag = 0;
        *odd_issued = 0;
        fence_mbar_init();
        for (int g = 0; g < batch.count; ++g) {
            tma_prefetch_desc(&batch.prob[g].map_a);
            tma_prefetch_desc(&batch.prob[g].map_b);
            if (EPI != EPI_F32) tma_prefetch_desc(&batch.prob[g].map_d);
            if (DSIG) tma_prefetch_desc(&batch.prob[g].map_z);
            if (EPI == EPI_GLU) {
                tma_prefetch_desc(&batch.prob[g].map_b2);
                tma_prefetch_desc(&batch.prob[g].map_d2);
                tma_prefetch_desc(&batch.prob[g].map_d3);
            }
        }
    }
    if (warp == 1) {
        if (PAIR) {
            tmem_alloc_pair(tmem_slot, C::TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(tmem_slot, C::TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    if (PAIR)
        cluster_sync();   // both CTAs' barriers initialised before any cross-CTA arrive
    else
        __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    // The prologue above overlaps the previous kernel's tail; global memory is
    // touched only after that kernel has completed.
    grid_dependency_wait();
    grid_launch_dependents();

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            long long issued = 0;
            bool ok = true;
            const int selftest = batch.prob[0].p.selftest;
            const bool no_loads = selftest == 1;
            const long long load_limit = (PAIR && !leader && selftest == 2) ? 1 : (1ll << 62);
            bool stop = false;
            WorkIter it;
            work_begin<EPI>(batch, first_unit, it);
            Unit x;
            while (ok && !stop && !no_loads && work_next<EPI>(batch, unit_step, it, x)) {
                const CUtensorMap* map_a = &batch.prob[x.g].map_a;
                const CUtensorMap* map_b = &batch.prob[x.g].map_b;
                // this CTA's rows of A and columns of B
                const int m0 = x.m_blk * TILE_M + static_cast<int>(rank) * C::CTA_ROWS;
                const int n0 = x.n_blk * BN + static_cast<int>(rank) * C::B_ROWS;
                for (int kb = x.kb0; kb < x.kb1; ++kb) {
                    if (issued >= load_limit) {
                        stop = true;
                        break;
                    }
                    if (!wait_bounded(&empty_bar[stage], phase ^ 1u, wc, ST_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sa = smem_a + stage * C::A_BYTES;
                    uint8_t* sb = smem_b + stage * C::B_BYTES;
                    const int k0 = kb * BK;
                    // EPI_GLU: the up half of the walk reads B_up from its own k = 0
                    int kB = k0;
                    const CUtensorMap* mb = map_b;
                    if (EPI == EPI_GLU && kb >= batch.prob[x.g].p.glu_half) {
                        kB = k0 - batch.prob[x.g].p.glu_half * BK;
                        mb = &batch.prob[x.g].map_b2;
                    }
                    if (PAIR) {
                        // both CTAs' boxes count on the even CTA's stage barrier
                        const uint32_t fb = mapa_shared(smem_u32(&full_bar[stage]), 0);
                        if (leader) mbar_arrive_expect_tx(&full_bar[stage], 2 * C::STAGE_BYTES);
                        if (A_MN) {
#pragma unroll
                            for (int j = 0; j < C::CTA_ROWS / 64; ++j)
                                tma_load_2d_pair(map_a, fb, sa + j * 64 * BK * 2, m0 + 64 * j, k0);
                        } else {
                            tma_load_2d_pair(map_a, fb, sa, k0, m0);
                        }
                        if (B_MN) {
#pragma unroll
                            for (int j = 0; j < C::B_ROWS / 64; ++j)
                                tma_load_2d_pair(mb, fb, sb + j * 64 * BK * 2, n0 + 64 * j, kB);
                        } else {
                            tma_load_2d_pair(mb, fb, sb, kB, n0);
                        }
                    } else {
                        mbar_arrive_expect_tx(&full_bar[stage], C::STAGE_BYTES);
                        if (A_MN) {                 // 64-row boxes along M
#pragma unroll
                            for (int j = 0; j < TILE_M / 64; ++j)
                                tma_load_2d(map_a, &full_bar[stage], sa + j * 64 * BK * 2, m0 + 64 * j, k0);
                        } else {                    // one box of TILE_M rows
                            tma_load_2d(map_a, &full_bar[stage], sa, k0, m0);
                        }
                        if (B_MN) {
#pragma unroll
                            for (int j = 0; j < BN / 64; ++j)
                                tma_load_2d(mb, &full_bar[stage], sb + j * 64 * BK * 2, n0 + 64 * j, kB);
                        } else {
                            tma_load_2d(mb, &full_bar[stage], sb, kB, n0);
                        }
                    }
                    ++issued;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // normal: every k-block of the walk issued, and the MMA warp has
            // released (its commits have arrived on) every stage since
            bool normal = ok && !*abort_flag;
            const int stage_end = stage;      // where the walk's last issue left the ring
            const uint32_t phase_end = phase;
            if (normal) {
                // tail: acquire every stage once more
                for (int j = 0; j < STAGES; ++j) {
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
            if (!normal && !PAIR) {
                // drain: the last min(issued, STAGES) loads may still be landing
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
            if (PAIR) {
                if (!leader) {
                    // report the k-blocks issued to the even CTA, whose stage barriers
                    // count them, and wait until it has seen every one of them land
                    st_shared_cluster_u32(mapa_shared(smem_u32(const_cast<int*>(odd_issued)), 0),
                                          static_cast<uint32_t>(issued));
                    mbar_arrive_cluster(mapa_shared(smem_u32(xchg_bar), 0));
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait_cluster(relay_bar, 0)) {
                        if (global_timer_ns() - t0 > 4 * WAIT_LIMIT_NS) {
                            if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                            break;
                        }
                    }
                } else {
                    bool got = true;
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait_cluster(xchg_bar, 0)) {
                        if (global_timer_ns() - t0 > 2 * WAIT_LIMIT_NS) {
                            if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                            got = false;
                            break;
                        }
                    }
                    if (got && !normal) {
                        // k-block q of the walk used stage q % STAGES in phase q / STAGES
                        const long long L = issued, O = *odd_issued;
                        const long long Q = L > O ? L : O;
                        for (long long q = O; q < L; ++q)   // the odd CTA's share will not come
                            mbar_complete_tx(&full_bar[q % STAGES], C::STAGE_BYTES);
                        for (long long q = L; q < Q; ++q)   // only the odd CTA's share is coming
                            mbar_arrive_expect_tx(&full_bar[q % STAGES], C::STAGE_BYTES);
                        for (long long q = Q > STAGES ? Q - STAGES : 0; q < Q; ++q) {
                            const uint64_t t1 = global_timer_ns();
                            while (!mbar_try_wait(&full_bar[q % STAGES], static_cast<uint32_t>((q / STAGES) & 1))) {
                                if (global_timer_ns() - t1 > WAIT_LIMIT_NS) {
                                    if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                                    break;
                                }
                            }
                        }
                    }
                    mbar_arrive_cluster(mapa_shared(smem_u32(relay_bar), 1));
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0 && leader) {   // a pair's MMAs are issued by its even CTA alone
            constexpr uint32_t idesc = idesc_bf16_f32(PAIR ? 2 * BM : BM, BN, A_MN ? 1 : 0, B_MN ? 1 : 0);
            int stage = 0;
            uint32_t phase = 0;
            int buf = 0;
            uint32_t bphase = 0;
            bool ok = true;
            bool issued_any = false;
            WorkIter it;
            work_begin<EPI>(batch, first_unit, it);
            Unit x;
            while (ok && work_next<EPI>(batch, unit_step, it, x)) {
                const int kb0 = x.kb0, kb1 = x.kb1;
                if (!wait_bounded<PAIR>(&tempty_bar[buf], bphase ^ 1u, wc, ST_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(GLU_SPLIT ? 0 : buf * C::ACC_COLS);
                // EPI_GLU: from k-block glu_half on, the up half accumulates into
                // the tile's second accumulator, starting afresh
                const int half = EPI == EPI_GLU ? batch.prob[x.g].p.glu_half : -1;
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (GLU_SPLIT && kb == half) {   // the up accumulator, freed by the previous tile's epilogue
                        if (!wait_bounded<PAIR>(&tempty_bar[1], bphase ^ 1u, wc, ST_TIMEOUT_MMA)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                    }
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
                        const uint64_t db = B_MN ? smem_desc_sw128(sb + ks * UMMA_K * 128, 64 * BK * 2, 1024)
                                                 : smem_desc_sw128(sb + ks * UMMA_K * 2, 16, 1024);
#pragma unroll
                        for (int sub = 0; sub < MSUB; ++sub) {
                            // sub-tile `sub` = A rows [128 sub, 128 sub + 128): +16 KB either way
                            const uint32_t sas = sa + sub * BM * BK * 2;
                            const uint64_t da = A_MN ? smem_desc_sw128(sas + ks * UMMA_K * 128, 64 * BK * 2, 1024)
                                                     : smem_desc_sw128(sas + ks * UMMA_K * 2, 16, 1024);
                            const bool second = EPI == EPI_GLU && kb >= half;
                            const uint32_t acc = (ks > 0 || (kb > kb0 && kb != half)) ? 1u : 0u;
                            const uint32_t d_acc = d_tmem + (second ? BN : 0);
                            if (PAIR)
                                umma_f16_pair(d_acc, da, db, idesc, acc);
                            else
                                umma_f16(d_acc + sub * BN, da, db, idesc, acc);
                        }
                    }
                    issued_any = true;
                    // frees the smem stage (of both CTAs of a pair) once these MMAs are done
                    if (PAIR)
                        umma_commit_pair(&empty_bar[stage], 0x3);
                    else
                        umma_commit(&empty_bar[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                // accumulator ready for the epilogue (of both CTAs of a pair)
                if (PAIR)
                    umma_commit_pair(&tfull_bar[buf], 0x3);
                else
                    umma_commit(&tfull_bar[buf]);
                if (GLU_SPLIT) {
                    bphase ^= 1u;   // one slot: buf stays 0
                } else if (++buf == 2) {
                    buf = 0;
                    bphase ^= 1u;
                }
            }
            if ((!ok || *abort_flag) && issued_any) {
                if (PAIR)
                    umma_commit_pair(drain_bar, 0x1);
                else
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
        // ------------------------------------------------ epilogue (warps 2..9)
        const int q = warp & 3;                 // TMEM lane quarter this warp may access
        const int half = (warp - 2) >> 2;       // which of the two warps on this quarter
        // MSUB == 2: each warp of a quarter owns one 128-row sub-tile and all its
        // chunks; MSUB == 1: the two warps take alternate chunks of the one sub-tile
        const int sub = (MSUB == 2) ? half : 0;
        const int c_first = (MSUB == 2) ? 0 : half;
        constexpr int C_STEP = (MSUB == 2) ? 1 : 2;
        const int row_off = PAIR ? static_cast<int>(rank) * BM : 0;   // this CTA's rows of a pair's tile
        const int row_in_tile = row_off + sub * BM + q * 32 + lane;
        uint8_t* ep_gen = smem_epi + (warp - 2) * EPI_WARP_BYTES;
        const uint32_t ep = smem_u32(ep_gen);
        uint64_t* zbar = zfull_bar + 2 * (warp - 2);
        int out_slot = 0;                       // next output box of the ring (EPI_STORE / EPI_ZH)
        int buf = 0;
        uint32_t bphase = 0;
        bool ok = true;

        // 32-column chunks of unit x that hold output rows of this warp
        auto chunk_count = [&](const Unit& x) {
            const GemmParams& pu = batch.prob[x.g].p;
            if (EPI == EPI_F32 || (EPI == EPI_TAIL && x.split >= 0)) return BN / 32;   // partial tiles: all of it
            if (x.m_blk * TILE_M + row_off + sub * BM + q * 32 >= pu.M) return 0;   // this warp's 32 rows are all past the end
            const int left = pu.N - x.n_blk * BN;
            return left >= BN ? BN / 32 : (left + 31) / 32;
        };
        int cur_M = 0;                          // output rows of the tile in hand

        // hand box `box` (already staged, fenced) to the TMA engine
        auto store_box = [&](const CUtensorMap* map, uint32_t box, int x, int y) {
            __syncwarp();
            if (lane == 0) {
                tma_store_2d(map, box, x, y);
                bulk_commit_group();
            }
        };
        // stage one output box (this thread's row) from the ring and store it
        auto emit = [&](const CUtensorMap* map, const uint32_t (&w)[16], int x, int y) {
            if (y >= cur_M) return;             // whole box below the last row: nothing to store
            const uint32_t box = ep + out_slot * EPI_BOX_BYTES;
            if (lane == 0) bulk_wait_group_read<EPI_OUT_BOXES - 1>();   // its previous store has read it
            __syncwarp();
            stage_row(box, lane, w);
            fence_proxy_async_smem();
            store_box(map, box, x, y);
            if (++out_slot == EPI_OUT_BOXES) out_slot = 0;
        };
        // store one 32-column chunk of a bf16 output (this thread's row) to the
        // tensor behind `map` (base `ptr`, pitch d_ld): through the box ring,
        // or, in the chunk that holds a ragged right edge, with masked direct
        // stores that leave the row padding untouched
        auto put = [&](const GemmParams& pp, const CUtensorMap* map, __nv_bfloat16* ptr, const uint32_t (&w)[16],
                       int col0, int row0, int row) {
            if ((pp.N & 7) != 0 && col0 + 32 > pp.N) {
                if (row < pp.M) {
                    uint16_t* d = reinterpret_cast<uint16_t*>(ptr + row * pp.d_ld + col0);
                    const int valid = pp.N - col0;
#pragma unroll
                    for (int j = 0; j < 32; ++j)   // fully unrolled: w stays in registers
                        if (j < valid) d[j] = static_cast<uint16_t>((j & 1) ? (w[j >> 1] >> 16) : (w[j >> 1] & 0xFFFFu));
                }
                return;
            }
            emit(map, w, col0, row0);
        };

        // EPI_DSIGMA: Z boxes run one (tile, chunk) item ahead of their use
        int zu = first_unit, zc = c_first;      // next item whose Z box is to be loaded
        uint32_t zphase = 0;                    // bit b: parity of the next wait on zbar[b]
        int zload = 0, zuse = 0;
        auto z_advance = [&]() {                // move (zu, zc) to the next item that has a chunk
            while (zu < batch.units && zc >= chunk_count(decode(batch, zu))) {
                zu += unit_step;
                zc = c_first;
            }
        };
        auto z_issue = [&]() {                  // load the Z box of item (zu, zc), then step past it
            if (zu >= batch.units) return;
            const Unit x = decode(batch, zu);
            const int b = zload & 1;
            if (lane == 0) {
                bulk_wait_group_read<0>();      // the stores that last read box b are done with it
                mbar_arrive_expect_tx(&zbar[b], EPI_BOX_BYTES);
                tma_load_2d(&batch.prob[x.g].map_z, &zbar[b], ep_gen + b * EPI_BOX_BYTES, x.n_blk * BN + zc * 32,
                            x.m_blk * TILE_M + row_off + sub * BM + q * 32);
            }
            ++zload;
            zc += C_STEP;
            z_advance();
        };
        if (DSIG) {
            z_advance();
            z_issue();
        }

        WorkIter it;
        work_begin<EPI>(batch, first_unit, it);
        Unit x;
        while (ok && work_next<EPI>(batch, unit_step, it, x)) {
            const GemmParams& p = batch.prob[x.g].p;
            const CUtensorMap* map_d = &batch.prob[x.g].map_d;
            const CUtensorMap* map_d2 = &batch.prob[x.g].map_d2;
            const int m_blk = x.m_blk, n_blk = x.n_blk, split = x.split;
            cur_M = p.M;
            const int row0 = m_blk * TILE_M + row_off + sub * BM + q * 32;
            const int row = row0 + lane;
            const int nch = chunk_count(x);
            if (!wait_bounded(&tfull_bar[buf], bphase, wc, ST_TIMEOUT_EPILOGUE)) break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>((GLU_SPLIT ? 0 : buf * C::ACC_COLS) + sub * BN);
            if constexpr (GLU_SPLIT) {
                // the gate half of this warp's chunks into registers, then free it
                uint32_t gsave[BN / 64][16];
#pragma unroll
                for (int i = 0; i < BN / 64; ++i) {
                    const int c = c_first + C_STEP * i;
                    if (c < nch) {
                        uint32_t v[32];
                        tmem_ld_32x32b_x32(tbase + c * 32, v);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            gsave[i][j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    }
                }
                tc_fence_before();
                if (PAIR)
                    mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[0]), 0));
                else
                    mbar_arrive(&tempty_bar[0]);
                // the up half: M = bf16(Y_gate * Y_up), and Y_gate, Y_up when training
#pragma unroll
                for (int i = 0; i < BN / 64; ++i) {
                    const int c = c_first + C_STEP * i;
                    if (c < nch) {
                        const int col0 = n_blk * BN + c * 32;
                        uint32_t v[32];
                        tmem_ld_32x32b_x32(tbase + BN + c * 32, v);
                        tmem_ld_wait();
                        uint32_t wu[16], w[16];
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            wu[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                            w[j] = pack_bf16x2(bf16_lo(gsave[i][j]) * bf16_lo(wu[j]), bf16_hi(gsave[i][j]) * bf16_hi(wu[j]));
                        }
                        put(p, map_d, p.d_ptr, w, col0, row0, row);
                        if (p.has_d2) {
                            put(p, map_d2, p.d2_ptr, gsave[i], col0, row0, row);
                            put(p, &batch.prob[x.g].map_d3, p.d3_ptr, wu, col0, row0, row);
                        }
                    }
                }
                tc_fence_before();
                if (PAIR)
                    mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[1]), 0));
                else
                    mbar_arrive(&tempty_bar[1]);
                bphase ^= 1u;
                continue;
            }
            if constexpr (EARLY_FREE) {
                // EPI_STORE, one 128-row sub-tile: this warp's chunks into
                // registers as bf16, the accumulator freed at once, then the
                // stores; the MMAs of the tile after next need not wait for the
                // stores of this one to drain through the box ring
                uint32_t wsave[BN / 64][16];
#pragma unroll
                for (int i = 0; i < BN / 64; ++i) {
                    const int c = c_first + C_STEP * i;
                    if (c < nch) {
                        uint32_t v[32];
                        tmem_ld_32x32b_x32(tbase + c * 32, v);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 16; ++j)
                            wsave[i][j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    }
                }
                tc_fence_before();
                if (PAIR)
                    mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[buf]), 0));
                else
                    mbar_arrive(&tempty_bar[buf]);
                if (++buf == 2) {
                    buf = 0;
                    bphase ^= 1u;
                }
#pragma unroll
                for (int i = 0; i < BN / 64; i += 2) {
                    const int c0 = c_first + C_STEP * i, c1 = c0 + C_STEP;
                    const bool full = c1 < nch && !((p.N & 7) != 0 && n_blk * BN + c1 * 32 + 32 > p.N) && row0 < cur_M;
                    if (full) {
                        // both boxes of the ring at once, behind one proxy fence
                        // (measured: the 1B Y GEMMs 3 %, the dX GEMMs 2 % faster
                        // than a fence per box)
                        if (lane == 0) bulk_wait_group_read<0>();
                        __syncwarp();
                        stage_row(ep, lane, wsave[i]);
                        stage_row(ep + EPI_BOX_BYTES, lane, wsave[i + 1]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(map_d, ep, n_blk * BN + c0 * 32, row0);
                            tma_store_2d(map_d, ep + EPI_BOX_BYTES, n_blk * BN + c1 * 32, row0);
                            bulk_commit_group();
                        }
                        out_slot = 0;
                    } else {
                        if (c0 < nch) put(p, map_d, p.d_ptr, wsave[i], n_blk * BN + c0 * 32, row0, row);
                        if (c1 < nch) put(p, map_d, p.d_ptr, wsave[i + 1], n_blk * BN + c1 * 32, row0, row);
                    }
                }
                continue;
            }
#pragma unroll 1
            for (int c = c_first; c < nch; c += C_STEP) {
                const int col0 = n_blk * BN + c * 32;
                if (DSIG) z_issue();   // the next item's Z box, while this one is processed
                // EPI_GLU_BWD: this row's Y_gate and Y_up chunk, loaded ahead of the accumulator
                uint4 yg[4], yu[4];
                if constexpr (EPI == EPI_GLU_BWD) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        yg[j] = yu[j] = make_uint4(0u, 0u, 0u, 0u);
                        if (row < p.M && col0 + 8 * j < p.N) {   // 8-column vectors inside the padded row
                            const long long off = static_cast<long long>(row) * p.d_ld + col0 + 8 * j;
                            yg[j] = __ldg(reinterpret_cast<const uint4*>(p.yg_ptr + off));
                            yu[j] = __ldg(reinterpret_cast<const uint4*>(p.yu_ptr + off));
                        }
                    }
                }
                uint32_t v[32];
                uint32_t v2[32];   // EPI_GLU: the same chunk of the up accumulator
                tmem_ld_32x32b_x32(tbase + c * 32, v);
                if constexpr (EPI == EPI_GLU) tmem_ld_32x32b_x32(tbase + BN + c * 32, v2);
                tmem_ld_wait();
                if (EPI == EPI_F32 || (EPI == EPI_TAIL && split >= 0)) {
                    float* dst = nullptr;
                    if (EPI == EPI_F32) {
                        if (row < p.M)              // rows past the last one: the reduce never reads them
                            dst = reinterpret_cast<float*>(p.D) + split * p.part_stride +
                                  static_cast<long long>(m_blk * TILE_M + row_in_tile) * p.ldd + col0;
                    } else {                        // the piece's partial slot: one whole TILE_M x BN tile
                        dst = batch.tail_part + static_cast<long long>(split) * (TILE_M * BN) +
                              static_cast<long long>(row_in_tile) * BN + c * 32;
                    }
                    if (dst) {
                        float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            d4[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                                __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
                    }
                    continue;
                }
                uint32_t w[16];
                if (EPI == EPI_STORE || EPI == EPI_TAIL) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    put(p, map_d, p.d_ptr, w, col0, row0, row);
                } else if (EPI == EPI_GLU) {
                    // Y_gate, Y_up rounded to bf16; M = bf16(Y_gate * Y_up) of the rounded
                    // values (their product is exact in fp32)
                    uint32_t wg[16], wu[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        wg[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                        wu[j] = pack_bf16x2(__uint_as_float(v2[2 * j]), __uint_as_float(v2[2 * j + 1]));
                        w[j] = pack_bf16x2(bf16_lo(wg[j]) * bf16_lo(wu[j]), bf16_hi(wg[j]) * bf16_hi(wu[j]));
                    }
                    put(p, map_d, p.d_ptr, w, col0, row0, row);
                    if (p.has_d2) {                 // training: Y_gate and Y_up for the backward
                        put(p, map_d2, p.d2_ptr, wg, col0, row0, row);
                        put(p, &batch.prob[x.g].map_d3, p.d3_ptr, wu, col0, row0, row);
                    }
                } else if (EPI == EPI_GLU_BWD) {
                    // dM rounded to bf16; dY_gate = bf16(dM * Y_up), dY_up = bf16(dM * Y_gate)
                    uint32_t dm[16], gw[16], uw[16];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        gw[4 * j] = yg[j].x;
                        gw[4 * j + 1] = yg[j].y;
                        gw[4 * j + 2] = yg[j].z;
                        gw[4 * j + 3] = yg[j].w;
                        uw[4 * j] = yu[j].x;
                        uw[4 * j + 1] = yu[j].y;
                        uw[4 * j + 2] = yu[j].z;
                        uw[4 * j + 3] = yu[j].w;
                    }
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        dm[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                        w[j] = pack_bf16x2(bf16_lo(dm[j]) * bf16_lo(uw[j]), bf16_hi(dm[j]) * bf16_hi(uw[j]));
                    }
                    put(p, map_d, p.d_ptr, w, col0, row0, row);      // dY_gate
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(bf16_lo(dm[j]) * bf16_lo(gw[j]), bf16_hi(dm[j]) * bf16_hi(gw[j]));
                    put(p, map_d2, p.d2_ptr, w, col0, row0, row);    // dY_up
                } else if (EPI == EPI_ZH) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        w[j] = pack_bf16x2(__uint_as_float(v[2 * j]), __uint_as_float(v[2 * j + 1]));
                    if (!p.h_only) emit(map_d, w, col0, row0);
                    if (p.has_d2 || p.h_only) {
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
                        emit(p.h_only ? map_d : map_d2, w, col0, row0);
                    }
                } else if (DSIG) {
                    const int b = zuse & 1;
                    const bool zok = wait_bounded(&zbar[b], (zphase >> b) & 1u, wc, ST_TIMEOUT_EPILOGUE);
                    zphase ^= 1u << b;
                    ++zuse;
                    if (!zok) {
                        ok = false;
                        break;
                    }
                    const uint32_t box = ep + b * EPI_BOX_BYTES;
                    uint32_t z[16];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const uint4 t = ld_shared_v4(box + box64_off(lane, j));
                        z[4 * j] = t.x;
                        z[4 * j + 1] = t.y;
                        z[4 * j + 2] = t.z;
                        z[4 * j + 3] = t.w;
                    }
                    if constexpr (EPI == EPI_DSIGMA_H) {
                        // CoLA-M: H = sigma(Z) formed with sigma'(Z), stored through the same box
                        uint32_t hw[16];
                        with_sigma_fixed<SIG>([&](auto tag) {
                            constexpr int S = decltype(tag)::value;
                            if constexpr (S == SIG_SILU) {
                                if (below_tanh_floor(z)) {
                                    dsilu_silu_chunk_fallback(z, v, w, hw);
                                    return;
                                }
                            }
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                float hl, dl, hh, dh;
                                act_both<S, LOGI_TANH>(bf16_lo(z[j]), hl, dl);
                                act_both<S, LOGI_TANH>(bf16_hi(z[j]), hh, dh);
                                w[j] = pack_bf16x2(__uint_as_float(v[2 * j]) * dl, __uint_as_float(v[2 * j + 1]) * dh);
                                hw[j] = pack_bf16x2(hl, hh);
                            }
                        });
                        stage_row(box, lane, w);    // dZ in place of this row's Z
                        fence_proxy_async_smem();
                        store_box(map_d, box, col0, row0);
                        if (lane == 0) bulk_wait_group_read<0>();
                        __syncwarp();
                        stage_row(box, lane, hw);
                        fence_proxy_async_smem();
                        store_box(map_d2, box, col0, row0);
                    } else {
                        with_sigma_fixed<SIG>([&](auto tag) {
                            constexpr int S = decltype(tag)::value;
                            if constexpr (S == SIG_SILU) {
                                if (below_tanh_floor(z)) {
                                    dsilu_chunk_fallback(z, v, w);
                                    return;
                                }
                            }
#pragma unroll
                            for (int j = 0; j < 16; ++j)
                                w[j] = pack_bf16x2(__uint_as_float(v[2 * j]) * act_dsigma<S, LOGI_TANH>(bf16_lo(z[j])),
                                                   __uint_as_float(v[2 * j + 1]) * act_dsigma<S, LOGI_TANH>(bf16_hi(z[j])));
                        });
                        stage_row(box, lane, w);    // dZ in place of this row's Z
                        fence_proxy_async_smem();
                        store_box(map_d, box, col0, row0);
                    }
                }
            }
            tc_fence_before();
            if (PAIR)   // the even CTA's barrier collects both CTAs' epilogues
                mbar_arrive_cluster(mapa_shared(smem_u32(&tempty_bar[buf]), 0));
            else
                mbar_arrive(&tempty_bar[buf]);
            if (++buf == 2) {
                buf = 0;
                bphase ^= 1u;
            }
        }
        // Z boxes still in flight (issued ahead, or for items the loop left early)
        while (zuse < zload) {
            const int b = zuse & 1;
            const uint64_t t0 = global_timer_ns();
            while (!mbar_try_wait(&zbar[b], (zphase >> b) & 1u)) {
                if (global_timer_ns() - t0 > WAIT_LIMIT_NS) {
                    if (status) atomicOr(status, ST_TIMEOUT_DRAIN);
                    break;
                }
            }
            zphase ^= 1u << b;
            ++zuse;
        }
        if (lane == 0) bulk_wait_group_all();   // every output store has landed
    }

    tc_fence_before();
    if (PAIR)
        cluster_sync();   // neither CTA leaves while the pair's MMAs may still read its shared memory
    else
        __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        if (PAIR)
            tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
        else
            tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

}  // namespace cola
