// host_plan.cuh -- host-side helpers shared by the ABI translation units:
// TMA descriptor encoding, GEMM tiling / token-split planning and the
// dispatch of a GEMM launch to its tile-width instantiation.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <mutex>

#include "gemm_launch.cuh"
#include "splitk_cluster.cuh"

namespace cola {
namespace {

// ------------------------------------------------------------ tensor maps
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn()
{
    static EncodeFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeFn>(p);
    });
    return fn;
}

// 2-D bf16 matrix [outer x inner] with row pitch ld (elements) and box
// {box_inner, box_outer}.  Loads read zeros outside the extents; stores are
// clipped to them.
bool make_map(CUtensorMap* m, const void* base, int64_t inner, int64_t outer, int64_t ld, int box_inner,
              int box_outer, CUtensorMapSwizzle swz)
{
    EncodeFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
    cuuint32_t box[2] = {static_cast<cuuint32_t>(box_inner), static_cast<cuuint32_t>(box_outer)};
    cuuint32_t estr[2] = {1u, 1u};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Epilogue box of 32 rows x 32 columns (64-byte rows, 64-byte swizzle): the
// unit in which the GEMM epilogue stores bf16 outputs and reads the saved Z.
bool map_box32(CUtensorMap* m, const void* base, int64_t cols, int64_t rows, int64_t ld)
{
    return make_map(m, base, cols, rows, ld, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B);
}

// K-major operand: rows are the M (or N) index, k contiguous: box {64, rows_per_tile}.
// MN-major operand: rows are k, the M (or N) index contiguous: box {64, 64}.
bool map_kmajor(CUtensorMap* m, const void* base, int64_t k_extent, int64_t mn_extent, int64_t ld, int tile_rows)
{
    return make_map(m, base, k_extent, mn_extent, ld, 64, tile_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

bool map_mnmajor(CUtensorMap* m, const void* base, int64_t mn_extent, int64_t k_extent, int64_t ld)
{
    return make_map(m, base, mn_extent, k_extent, ld, 64, 64, CU_TENSOR_MAP_SWIZZLE_128B);
}

// ------------------------------------------------------------ planning
// Column tile: the width that pads N least; a compute-heavy GEMM (see
// heavy_gemm) takes 256 whenever that pads N by at most 5 %, because only
// 256-column tiles run on CTA pairs.
int choose_bn(int64_t N, bool heavy = false)
{
    if (N <= 128) return 128;
    const int64_t pad256 = (N + 255) / 256 * 256;
    const int64_t pad128 = (N + 127) / 128 * 128;
    if (heavy && N >= 1024 && pad256 * 100 <= N * 105) return 256;
    return pad256 <= pad128 ? 256 : 128;
}

// Compute-heavy: more than one 128-row block and either >= 64 GFLOP, or
// >= 16 GFLOP at an arithmetic intensity (each operand read once, the
// result written once) of >= 300 FLOP/B, above the ridge of the GB300 bf16
// roofline (~287).  The second clause takes the tensor-bound GEMMs of the
// 8192-token inference workloads (measured: 1B forward -14 %).
bool heavy_gemm(int64_t M, int64_t N, int64_t K)
{
    const double m = static_cast<double>(M), n = static_cast<double>(N), k = static_cast<double>(K);
    const double flops = 2.0 * m * n * k;
    const double bytes = 2.0 * (m * k + n * k + m * n);
    return M > 128 && (flops >= 64e9 || (flops >= 16e9 && flops / bytes >= 300.0));
}

// A GEMM of one 128-row block (a few tokens: decode) streams its B operand
// through as many CTAs as it has column tiles, so it takes 128-column tiles:
// twice the CTAs of 256-column ones, up to N = 8192 (64 tiles; wider ones,
// often batched in twos, would spill into a second wave of CTAs).  Measured:
// 1B decode step 0.066 -> 0.059 ms, 7B 0.090 -> 0.081 ms.
int choose_bn_for(int64_t M, int64_t N, int64_t K)
{
    if (M <= 128 && N <= 8192) return 128;
    return choose_bn(N, heavy_gemm(M, N, K));
}

// Tile modes ("msub" below): 1 = one CTA runs a 128-row tile; 2 = one CTA
// runs two 128-row sub-tiles sharing each B tile; TILE_PAIR = a CTA pair runs
// a 256-row tile with tcgen05 cta_group::2 (each CTA loads half of B).
constexpr int TILE_PAIR = 3;

int tile_rows(int msub) { return msub == 1 ? BM : 2 * BM; }        // rows of one unit
int a_box_rows(int msub) { return msub == TILE_PAIR ? BM : BM * msub; }   // rows of A one CTA loads
int b_box_rows(int bn, int msub) { return msub == TILE_PAIR ? bn / 2 : bn; }   // K-major B rows one CTA loads
int unit_slots(int msub, int sms) { return msub == TILE_PAIR ? sms / 2 : sms; }   // units in flight

// Compute-heavy GEMMs with 256-column tiles and K >= 512 run on CTA pairs:
// halving each CTA's B traffic relieves the shared-memory bandwidth that a
// single CTA's M = 128 MMAs, its TMA fills and its epilogue stores saturate
// (measured: -5 to -25 % per GEMM on the 1B layers, K = 512 to 65536).  With
// K = 256 (4 k-blocks per tile, the store-bound Y and dX GEMMs at rank 256)
// a pair was 20-40 % slower, and with 128-column tiles slower than one CTA
// running two 128-row sub-tiles (+12 to +23 %), which those keep.  The
// HBM-bound short GEMMs keep single-CTA 128-row tiles (a taller tile
// lengthens the epilogue they are limited by).
int choose_msub(int64_t M, int64_t N, int64_t K, int bn)
{
    if (!heavy_gemm(M, N, K)) return 1;
    if (bn == 256) return K >= 512 ? TILE_PAIR : 1;
    return 2;
}

// Tile grid of one GEMM, without a token split.
GemmParams base_params(int64_t M, int64_t N, int64_t K, int bn, int msub)
{
    GemmParams p;
    std::memset(&p, 0, sizeof p);
    p.M = static_cast<int>(M);
    p.N = static_cast<int>(N);
    p.k_blocks = static_cast<int>((K + BK - 1) / BK);
    p.m_tiles = static_cast<int>((M + tile_rows(msub) - 1) / tile_rows(msub));
    p.n_tiles = static_cast<int>((N + bn - 1) / bn);
    p.kb_per_split = p.k_blocks;
    p.splits = 1;
    p.units = p.m_tiles * p.n_tiles;
    return p;
}

// Token split of weight-gradient GEMMs sharing one launch (same K): minimise
// (waves of persistent CTAs) x (k-blocks per unit + the cost of writing and
// re-reading its fp32 partial tile, counted in k-blocks of operand bytes:
// 8 BN rows / (128 (rows + BN)), plus 2 for the reduction pass), with at least
// 4 k-blocks per split.
int choose_splits(int tiles, int k_blocks, int bn, int msub, int sms)
{
    const int max_s = k_blocks / 4 > 1 ? k_blocks / 4 : 1;
    const int rows = tile_rows(msub);
    const double c_part = 8.0 * bn * rows / (128.0 * (rows + bn)) + 2.0;
    sms = unit_slots(msub, sms);
    double best = -1.0;
    int S = 1;
    for (int s = 1; s <= max_s; ++s) {
        const long long units = static_cast<long long>(tiles) * s;
        const long long waves = (units + sms - 1) / sms;
        const long long kb = (k_blocks + s - 1) / s;
        const double cost = static_cast<double>(waves) * (static_cast<double>(kb) + (s > 1 ? c_part : 0.0));
        if (best < 0 || cost < best) {
            best = cost;
            S = s;
        }
    }
    return S;
}

void set_splits(GemmParams& p, int S)
{
    p.kb_per_split = (p.k_blocks + S - 1) / S;
    p.splits = (p.k_blocks + p.kb_per_split - 1) / p.kb_per_split;
    p.units = p.m_tiles * p.n_tiles * p.splits;
}

// Split-K for the forward GEMMs of small launches: with fewer output tiles
// than half the SMs (a few hundred tokens or less) and K >= 1024, the K range
// of each tile is split (>= 4 k-blocks per split, up to about one unit per
// SM); the fp32 partials are reduced, and the epilogue applied, by the reduce
// kernel.  A shorter K streams too little per tile for the extra reduce
// launch to pay off (measured: the 2048-token 60M layer, K = 512 / 128, got
// slower).  1 = no split.
int small_launch_splits(int tiles, int k_blocks, int sms)
{
    if (2 * tiles >= sms || k_blocks < 16) return 1;
    const int s = (sms + tiles - 1) / tiles;
    return s < k_blocks / 4 ? s : k_blocks / 4;
}

// K splits of a small launch reduced inside thread-block clusters
// (splitk_cluster.cuh, 128 x 128 tiles): with fewer tiles than half the SMs,
// the largest S <= 8 that keeps tiles * S within the SMs and >= 4 k-blocks
// per split.  1 = no split.
int cluster_splits(int tiles, int k_blocks, int sms)
{
    if (tiles < 1 || 2 * tiles >= sms) return 1;
    int s = sms / tiles;
    if (s > MAX_CLUSTER) s = MAX_CLUSTER;
    if (s > k_blocks / 4) s = k_blocks / 4;
    return s < 1 ? 1 : s;
}

int64_t partial_elems(const GemmParams& p, int bn, int msub)
{
    return static_cast<int64_t>(p.m_tiles) * tile_rows(msub) * p.n_tiles * bn;
}

// Weight-gradient group plan: count GEMMs D_i[M_i x N_i] = sum over the same
// ntok tokens, run by one launch with one tile configuration and one split.
struct WgradPlan {
    int bn, msub, splits, count;
    GemmParams p[MAX_GROUP];
    int64_t slab[MAX_GROUP];       // fp32 elements per split slab of each GEMM
    int64_t part_elems;            // all slabs of all splits
    double cost;                   // choose_splits' cost of the chosen split
};

WgradPlan plan_wgrad(const int64_t* M, const int64_t* N, int count, int64_t ntok, int sms)
{
    WgradPlan w;
    std::memset(&w, 0, sizeof w);
    w.count = count;
    w.bn = 256;
    for (int i = 0; i < count; ++i) {
        const int b = choose_bn_for(M[i], N[i], ntok);
        w.bn = b < w.bn ? b : w.bn;
    }
    w.msub = TILE_PAIR;   // the smallest tile any GEMM of the group would take
    for (int i = 0; i < count; ++i) {
        const int ms = choose_msub(M[i], N[i], ntok, w.bn);
        if (ms == 1 || (ms == 2 && w.msub == TILE_PAIR)) w.msub = ms;
    }
    int tiles = 0;
    for (int i = 0; i < count; ++i) {
        w.p[i] = base_params(M[i], N[i], ntok, w.bn, w.msub);
        // the token-major operands are read along the whole reduction: walk
        // the tiles so that a wave shares the panels of the larger one
        w.p[i].n_major = N[i] > M[i] ? 1 : 0;
        tiles += w.p[i].m_tiles * w.p[i].n_tiles;
    }
    const int S = choose_splits(tiles, w.p[0].k_blocks, w.bn, w.msub, sms);
    w.part_elems = 0;
    for (int i = 0; i < count; ++i) {
        set_splits(w.p[i], S);
        w.slab[i] = partial_elems(w.p[i], w.bn, w.msub);
        w.part_elems += static_cast<int64_t>(w.p[i].splits) * w.slab[i];
    }
    w.splits = w.p[0].splits;
    {
        const int rows = tile_rows(w.msub);
        const double c_part = 8.0 * w.bn * rows / (128.0 * (rows + w.bn)) + 2.0;
        const int sl = unit_slots(w.msub, sms);
        const long long units = static_cast<long long>(tiles) * w.splits;
        const long long waves = (units + sl - 1) / sl;
        w.cost = static_cast<double>(waves) * (w.p[0].kb_per_split + (w.splits > 1 ? c_part : 0.0));
    }
    return w;
}

// Split-tail schedule of a weight-gradient launch with bf16 outputs
// (EPI_TAIL).  The output tiles run whole in waves of `slots` CTAs (CTA
// pairs); the CTAs of a wave walk the token range in step, so the operand
// panels their tiles share are read from HBM about once.  The R < slots
// tiles of the last, partial wave are split over the tokens into `pieces`
// pieces each (R x pieces <= slots, >= 4 k-blocks per piece), so that the
// last wave is as short as the others allow; the tail reduce sums their
// partial slots.  Only the tail tiles write fp32 partials.  (Walking every
// CTA's equal share of all tile-and-token steps instead, stream-K style, was
// measured 1.4 to 1.6x slower at 60M to 7B: the CTAs drift apart in the token
// range, and the shared panels are then read from HBM once per tile.)
struct TailPlan {
    int body;                  // whole tiles (full waves)
    int tail;                  // tiles of the last wave
    int ntiles;                // tail tiles the reduce finishes (tail when split, else 0)
    int pieces, kps;           // pieces per tail tile, k-blocks per piece
    int units;                 // body + ntiles x pieces
    int kb;
    int tile_begin[MAX_GROUP];
    int64_t part_elems;        // ntiles x pieces x tile_rows x bn fp32 (0 when pieces == 1)
    double cost;               // k-blocks of the busiest CTA, plus the partial round trip
    TailTile tile[MAX_TAIL_TILES];
};

TailPlan plan_tail(const GemmParams* p, int count, int bn, int msub, int sms)
{
    TailPlan s;
    std::memset(&s, 0, sizeof s);
    int tiles = 0;
    for (int g = 0; g < count; ++g) {
        s.tile_begin[g] = tiles;
        tiles += p[g].m_tiles * p[g].n_tiles;
    }
    s.kb = p[0].k_blocks;
    const int slots = unit_slots(msub, sms);
    const int waves = tiles / slots;
    const int R = tiles - waves * slots;
    s.body = waves * slots;
    s.tail = R;
    s.pieces = 1;
    s.kps = s.kb;
    if (R > 0 && R <= MAX_TAIL_TILES) {
        const int most = s.kb / 4 > 1 ? s.kb / 4 : 1;
        int St = slots / R < most ? slots / R : most;
        if (St > 1) {
            s.kps = (s.kb + St - 1) / St;
            St = (s.kb + s.kps - 1) / s.kps;   // no empty piece
        }
        s.pieces = St > 1 ? St : 1;
        if (s.pieces == 1) s.kps = s.kb;
    }
    s.units = s.body + R * s.pieces;
    const int rows = tile_rows(msub);
    const double c_part = 8.0 * bn * rows / (128.0 * (rows + bn)) + 2.0;   // as in choose_splits
    s.cost = static_cast<double>(waves) * s.kb + (R > 0 ? s.kps + (s.pieces > 1 ? c_part : 0.0) : 0.0);
    if (s.pieces > 1) {
        s.part_elems = static_cast<int64_t>(R) * s.pieces * rows * bn;
        s.ntiles = R;
        for (int i = 0; i < R; ++i) {
            const int t = s.body + i;
            int g = 0;
            for (int j = 1; j < count; ++j)
                if (t >= s.tile_begin[j]) g = j;
            int mb = 0, nb = 0;
            tile_coords(p[g], t - s.tile_begin[g], mb, nb);
            TailTile& e = s.tile[i];
            e.g = g;
            e.m0 = mb * rows;
            e.n0 = nb * bn;
            e.lo_slot = i * s.pieces;
            e.count = s.pieces;
        }
    }
    return s;
}

// The tile configuration dispatch() launches for a planned (bn, msub): bit 2
// set when the launch runs on CTA pairs (clusters of two, cta_group::2), bit
// 3 when one CTA runs two 128-row sub-tiles.  These are the launch-trace
// flag bits of the same meaning (include/cola.h).
constexpr int TRACE_PAIR = 4;
constexpr int TRACE_MSUB2 = 8;
constexpr int TRACE_TAIL = 16;   // weight gradients with a split tail
constexpr int TRACE_GLU = 32;    // the dX epilogue stored the gated-MLP gradients dY_gate, dY_up
constexpr int TRACE_Z = 64;      // the fused forward stored Z
constexpr int TRACE_CLUSTER = 128;   // K splits reduced inside thread-block clusters (no reduce launch)

template <bool A_MN, int EPI>
int tile_flags(int bn, int msub)
{
    constexpr bool small_only = EPI == EPI_F32 && !A_MN;   // split-K forward partials: 128-row tiles only
    if (small_only) return 0;
    if (msub == TILE_PAIR && bn == 256) return TRACE_PAIR;
    if (msub == 2 && bn == 128) return TRACE_MSUB2;
    return 0;
}

// Launch one batch (all problems of one configuration).  Programmatic
// dependent launch hides launch latency and the prologue of short GEMMs
// (measured: -8 % step time on the HBM-bound 60M block) but costs ~1 % on
// long ones, so it is used below 64 GFLOP per launch.
template <bool A_MN, bool B_MN, int EPI, int SIG>
cudaError_t dispatch_sig(int bn, int msub, GemmBatch& b, int sms, cudaStream_t s)
{
    double flops = 0.0;
    int units = 0;
    for (int g = 0; g < b.count; ++g) {
        b.prob[g].unit_begin = units;
        units += b.prob[g].p.units;
        flops += 2.0 * b.prob[g].p.M * b.prob[g].p.N * (static_cast<double>(b.prob[g].p.k_blocks) * BK);
    }
    if constexpr (EPI == EPI_TAIL) units = b.tail_body + b.tail_tiles * b.tail_pieces;
    b.units = units;
    const bool pdl = flops < 64e9;
    // the split-K forward GEMMs of small launches (K-major fp32 partials) run
    // on single-CTA 128-row tiles only
    constexpr bool small_only = EPI == EPI_F32 && !A_MN;
    if constexpr (!small_only) {
        if (msub == TILE_PAIR && bn == 256) {
            const int pairs = units < sms / 2 ? units : sms / 2;
            return launch_gemm<256, 1, A_MN, B_MN, EPI, true, SIG>(b, 2 * pairs, pdl, s);
        }
    }
    if (msub != 1 && (bn == 256 || small_only)) return cudaErrorInvalidValue;   // planned tiles exist as above only
    const int grid = units < sms ? units : sms;
    if (bn == 256) return launch_gemm<256, 1, A_MN, B_MN, EPI, false, SIG>(b, grid, pdl, s);
    if constexpr (!small_only) {
        if (msub != 1) return launch_gemm<128, 2, A_MN, B_MN, EPI, false, SIG>(b, grid, pdl, s);
    }
    return launch_gemm<128, 1, A_MN, B_MN, EPI, false, SIG>(b, grid, pdl, s);
}

// The launch of a batch whose epilogue applies sigma (EPI_ZH, EPI_DSIGMA,
// EPI_DSIGMA_H) goes to the kernel compiled for its activation (the problems
// of one batch share it); the other kinds have one kernel.
template <bool A_MN, bool B_MN, int EPI>
cudaError_t dispatch(int bn, int msub, GemmBatch& b, int sms, cudaStream_t s)
{
    if constexpr (EPI == EPI_ZH || EPI == EPI_DSIGMA || EPI == EPI_DSIGMA_H) {
        switch (b.prob[0].p.sigma) {
        case SIG_SILU: return dispatch_sig<A_MN, B_MN, EPI, SIG_SILU>(bn, msub, b, sms, s);
        case SIG_GELU: return dispatch_sig<A_MN, B_MN, EPI, SIG_GELU>(bn, msub, b, sms, s);
        case SIG_IDENTITY: return dispatch_sig<A_MN, B_MN, EPI, SIG_IDENTITY>(bn, msub, b, sms, s);
        default: return cudaErrorInvalidValue;
        }
    } else {
        return dispatch_sig<A_MN, B_MN, EPI, SIG_IDENTITY>(bn, msub, b, sms, s);
    }
}

// The gated-MLP forward launch (EPI_GLU) with `bn`-column tiles: on CTA
// pairs (when `pair`) either 256 x 256 tiles with one TMEM slot whose gate and
// up accumulators are freed apart, or 256 x 128 tiles with two
// double-buffered slots; 128 x 128 tiles on single CTAs.
cudaError_t dispatch_glu(int bn, bool pair, GemmBatch& b, int sms, cudaStream_t s)
{
    b.prob[0].unit_begin = 0;
    b.units = b.prob[0].p.units;
    const GemmParams& p = b.prob[0].p;
    const bool pdl = 2.0 * p.M * p.N * (static_cast<double>(p.k_blocks) * BK) < 64e9;
    if (pair) {
        const int pairs = b.units < sms / 2 ? b.units : sms / 2;
        if (bn == 256) return launch_gemm<256, 1, false, false, EPI_GLU, true>(b, 2 * pairs, pdl, s);
        return launch_gemm<128, 1, false, false, EPI_GLU, true>(b, 2 * pairs, pdl, s);
    }
    return launch_gemm<128, 1, false, false, EPI_GLU>(b, b.units < sms ? b.units : sms, pdl, s);
}

}  // namespace
}  // namespace cola
