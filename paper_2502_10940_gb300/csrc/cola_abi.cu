// cola_abi.cu -- the extern "C" entry points of libcola.so (declared in
// include/cola.h): argument validation, workspace layout, TMA descriptors and
// the launch sequence of each pass of the CoLA layer.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "cola.h"
#include "fused_layer.cuh"
#include "gemm_launch.cuh"
#include "host_plan.cuh"

namespace cola {
namespace {

// ------------------------------------------------------------ device info
// Queried once per device; `ok` is published (release) after `sms`, so a
// thread that reads ok != 0 without the lock also sees sms.
struct DevInfo {
    std::atomic<int> ok{0};   // 1: queried, 2: unsupported device
    int sms = 0;
};

DevInfo g_dev[64];
std::mutex g_mu;

cola_status_t device_info(int* sms)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return COLA_ERR_LAUNCH;
    DevInfo& d = g_dev[dev];
    int ok = d.ok.load(std::memory_order_acquire);
    if (ok == 0) {
        std::lock_guard<std::mutex> lock(g_mu);
        ok = d.ok.load(std::memory_order_relaxed);
        if (ok == 0) {
            int major = 0, minor = 0, n = 0;
            if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
                return COLA_ERR_LAUNCH;
            d.sms = n;
            ok = (major == 10 && minor == 3) ? 1 : 2;   // kernels are built for sm_103a only
            d.ok.store(ok, std::memory_order_release);
        }
    }
    if (ok != 1) return COLA_ERR_UNSUPPORTED;
    *sms = d.sms;
    return COLA_OK;
}

// ------------------------------------------------------------ validation
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Shape {
    int64_t n, d_in, d_out, r, ld_x, ld_y, ld_a;
};

cola_status_t check_desc(const cola_desc_t* d, Shape* s)
{
    if (!d) return COLA_ERR_INVALID;
    if (d->n < 1 || d->d_in < 1 || d->d_out < 1 || d->r < 1) return COLA_ERR_INVALID;
    if (d->sigma < COLA_SIGMA_IDENTITY || d->sigma > COLA_SIGMA_GELU) return COLA_ERR_INVALID;
    if (d->mode != COLA_MODE_COLA && d->mode != COLA_MODE_COLA_M && d->mode != COLA_MODE_INFER)
        return COLA_ERR_INVALID;
    if (d->wgrad_fp32 != 0 && d->wgrad_fp32 != 1) return COLA_ERR_INVALID;
    if (d->reserved != 0) return COLA_ERR_INVALID;
    if (d->r % 64 != 0) return COLA_ERR_UNSUPPORTED;
    s->n = d->n;
    s->d_in = d->d_in;
    s->d_out = d->d_out;
    s->r = d->r;
    s->ld_x = d->ld_x ? d->ld_x : d->d_in;
    s->ld_y = d->ld_y ? d->ld_y : d->d_out;
    s->ld_a = d->ld_a ? d->ld_a : d->d_in;
    if (s->ld_x < s->d_in || s->ld_y < s->d_out || s->ld_a < s->d_in) return COLA_ERR_INVALID;
    if (s->ld_x % 8 || s->ld_y % 8 || s->ld_a % 8) return COLA_ERR_INVALID;
    const int64_t lim = (int64_t(1) << 31) - 256;
    if (s->n > lim || s->d_in > lim || s->d_out > lim || 3 * s->r > lim || s->ld_x > lim || s->ld_y > lim ||
        s->ld_a > lim)
        return COLA_ERR_UNSUPPORTED;
    // the work units of one launch are numbered in 32 bits: up to 3 projections
    // of (n / 128) x (width / 128) output tiles, or up to 4 weight gradients of
    // (width / 128)^2 tiles split up to n / 256 ways
    const double w = static_cast<double>(std::max({s->d_in, s->d_out, 3 * s->r}));
    const double row_tiles = std::ceil(static_cast<double>(s->n) / 128.0), col_tiles = std::ceil(w / 128.0);
    const double cap = 2147483647.0 / 2.0;
    if (3.0 * row_tiles * col_tiles > cap || 4.0 * col_tiles * col_tiles * std::ceil(s->n / 256.0) > cap)
        return COLA_ERR_UNSUPPORTED;
    return COLA_OK;
}

cola_status_t check_ptrs(std::initializer_list<const void*> required)
{
    for (const void* p : required) {
        if (!p) return COLA_ERR_INVALID;
        if (!aligned16(p)) return COLA_ERR_ALIGN;
    }
    return COLA_OK;
}

// The saved activations a forward call is given: Z under the training modes,
// H under CoLA only, neither under inference.
cola_status_t check_saved(int mode, const void* Z, const void* H)
{
    const bool want_z = mode != COLA_MODE_INFER;
    const bool want_h = mode == COLA_MODE_COLA;
    if ((Z != nullptr) != want_z || (H != nullptr) != want_h) return COLA_ERR_INVALID;
    if ((Z && !aligned16(Z)) || (H && !aligned16(H))) return COLA_ERR_ALIGN;
    return COLA_OK;
}

// ------------------------------------------------------------ workspace
constexpr size_t WS_HEADER = 256;
constexpr size_t WS_ALIGN = 256;

size_t align_up(size_t v) { return (v + WS_ALIGN - 1) / WS_ALIGN * WS_ALIGN; }

struct WsLayout {
    size_t dz_off, h_off, part_off, total;
};

// The weight-gradient group of one backward call: dB (per projection) and dA,
// all reduced over the same n tokens in one launch.
WgradPlan wgrad_plan(const cola_desc_t& d, int nproj, int sms)
{
    const int64_t R = nproj * d.r;
    int64_t M[MAX_GROUP], N[MAX_GROUP];
    const int nb = nproj;
    for (int j = 0; j < nb; ++j) {
        M[j] = d.d_out;
        N[j] = d.r;
    }
    M[nb] = R;
    N[nb] = d.d_in;
    return plan_wgrad(M, N, nb + 1, d.n, sms);
}

// The split-tail schedule of the same group (bf16 gradients): the tile
// configuration of wgrad_plan.  It runs when its cost is no higher than the
// uniform token split's (tail_wins).
TailPlan wgrad_tail_plan(const WgradPlan& w, int64_t ntok, int sms)
{
    GemmParams p[MAX_GROUP];
    for (int j = 0; j < w.count; ++j) {
        p[j] = base_params(w.p[j].M, w.p[j].N, ntok, w.bn, w.msub);
        p[j].n_major = w.p[j].n_major;
    }
    return plan_tail(p, w.count, w.bn, w.msub, sms);
}

bool tail_wins(const WgradPlan& w, const TailPlan& t) { return t.cost <= w.cost; }

// fp32 partial elements the forward of `nproj` projections needs when its
// GEMMs are small enough to be split over K (small_launch_splits)
int64_t fwd_part_elems(const cola_desc_t& d, int nproj, int sms)
{
    int64_t need = 0;
    const int64_t R = nproj * d.r;
    const int bn1 = choose_bn_for(d.n, R, d.d_in);
    if (choose_msub(d.n, R, d.d_in, bn1) == 1) {
        GemmParams p = base_params(d.n, R, d.d_in, bn1, 1);
        const int S = small_launch_splits(p.m_tiles * p.n_tiles, p.k_blocks, sms);
        if (S > 1) {
            set_splits(p, S);
            need = std::max<int64_t>(need, p.splits * partial_elems(p, bn1, 1));
        }
    }
    const int bn2 = choose_bn_for(d.n, d.d_out, d.r);
    if (choose_msub(d.n, d.d_out, d.r, bn2) == 1) {
        GemmParams p = base_params(d.n, d.d_out, d.r, bn2, 1);
        const int S = small_launch_splits(nproj * p.m_tiles * p.n_tiles, p.k_blocks, sms);
        if (S > 1) {
            set_splits(p, S);
            need = std::max<int64_t>(need, nproj * p.splits * partial_elems(p, bn2, 1));
        }
    }
    return need;
}

// dZ [n x R] bf16 (training modes), H [n x R] bf16 (CoLA-M and inference),
// the fp32 split partials of the weight-gradient group (training modes).
WsLayout ws_layout(const cola_desc_t& d, int nproj, int sms)
{
    const int64_t R = nproj * d.r;
    WsLayout L;
    size_t off = WS_HEADER;
    L.dz_off = off;
    if (d.mode != COLA_MODE_INFER) off += align_up(static_cast<size_t>(d.n) * R * 2);
    L.h_off = off;
    if (d.mode != COLA_MODE_COLA) off += align_up(static_cast<size_t>(d.n) * R * 2);
    L.part_off = off;
    // fp32 partials: of the split-K forward GEMMs of small launches, or of the
    // weight gradients (the forward and backward calls use them in turn)
    size_t part = static_cast<size_t>(fwd_part_elems(d, nproj, sms)) * 4;
    if (d.mode != COLA_MODE_INFER) {
        const WgradPlan w = wgrad_plan(d, nproj, sms);
        const TailPlan t = wgrad_tail_plan(w, d.n, sms);
        if (!d.wgrad_fp32 && tail_wins(w, t))
            part = std::max(part, static_cast<size_t>(t.part_elems) * 4);
        else
            part = std::max(part, static_cast<size_t>(w.part_elems) * 4);
    }
    off += align_up(part);
    L.total = off;
    return L;
}

cola_status_t check_ws(const cola_desc_t& d, int nproj, int sms, void* ws, size_t ws_bytes, WsLayout* L)
{
    if (!ws) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    *L = ws_layout(d, nproj, sms);
    if (ws_bytes < L->total) return COLA_ERR_WORKSPACE;
    return COLA_OK;
}

inline cola_status_t launched(cudaError_t e) { return e == cudaSuccess ? COLA_OK : COLA_ERR_LAUNCH; }

#define COLA_TRY(expr)                          \
    do {                                        \
        cola_status_t _st = (expr);             \
        if (_st != COLA_OK) return _st;         \
    } while (0)

#define COLA_MAP(expr)                          \
    do {                                        \
        if (!(expr)) return COLA_ERR_LAUNCH;    \
    } while (0)

uint8_t* wsb(void* ws) { return static_cast<uint8_t*>(ws); }
unsigned int* ws_status(void* ws) { return static_cast<unsigned int*>(ws); }

// ------------------------------------------------------------ launch tracing
struct TraceState {
    cola_trace_slot_t* slots = nullptr;
    int32_t capacity = 0;
    int32_t* count = nullptr;
};
TraceState g_trace;

// Launch through `fn`, bracketed by the next free trace slot's events.
template <class Fn>
cudaError_t traced(int kind, int count, const int64_t (*mnk)[3], int splits, int flags, cudaStream_t st, Fn&& fn)
{
    cola_trace_slot_t* slot = nullptr;
    if (g_trace.slots && g_trace.count && *g_trace.count >= 0 && *g_trace.count < g_trace.capacity)
        slot = &g_trace.slots[*g_trace.count];
    cudaError_t e;
    if (slot && (e = cudaEventRecord(static_cast<cudaEvent_t>(slot->start), st)) != cudaSuccess) return e;
    if ((e = fn()) != cudaSuccess) return e;
    if (slot) {
        if ((e = cudaEventRecord(static_cast<cudaEvent_t>(slot->stop), st)) != cudaSuccess) return e;
        slot->kernel = kind;
        slot->count = count;
        for (int g = 0; g < MAX_GROUP; ++g)
            for (int j = 0; j < 3; ++j) slot->mnk[g][j] = g < count ? static_cast<int32_t>(mnk[g][j]) : 0;
        slot->splits = splits;
        slot->flags = flags;
        ++*g_trace.count;
    }
    return cudaSuccess;
}

// Launch a batch of `count` problems of one configuration, traced as one
// launch; `tail` (EPI_TAIL only) is its split-tail schedule, with the
// partial slots at tail_part.
template <bool A_MN, bool B_MN, int EPI>
cola_status_t run_batch(int kind, int bn, int msub, const GemmProblem* probs, const int64_t (*mnk)[3], int count,
                        int flags, int sms, cudaStream_t st, const TailPlan* tail = nullptr, float* tail_part = nullptr)
{
    GemmBatch b;
    std::memset(&b, 0, sizeof b);
    b.count = count;
    for (int g = 0; g < count; ++g) b.prob[g] = probs[g];
    int splits = probs[0].p.splits;
    if (tail) {
        b.tail_body = tail->body;
        b.tail_tiles = tail->tail;
        b.tail_pieces = tail->pieces;
        b.tail_kps = tail->kps;
        for (int g = 0; g < count; ++g) b.tile_begin[g] = tail->tile_begin[g];
        b.tail_part = tail_part;
        flags |= TRACE_TAIL;
        splits = tail->pieces;
    }
    flags |= tile_flags<A_MN, EPI>(bn, msub);
    return launched(traced(kind, count, mnk, splits, flags, st,
                           [&] { return dispatch<A_MN, B_MN, EPI>(bn, msub, b, sms, st); }));
}

// ------------------------------------------------------------ passes
}  // namespace

cudaError_t launch_splitk_cluster(const CredBatch& b, bool pdl, cudaStream_t stream);

namespace {

// Whether weight-gradient launches of few tiles split the tokens inside
// thread-block clusters (cola_set_cluster_splitk); off: the planned split
// with its reduce launch.
std::atomic<int> g_cluster_splitk{1};

// One gradient of a cluster-reduced launch: D [M x N] = sum over the tokens
// of P[t, m] Q[t, n], both token-major (pitches ldp, ldq), D with pitch ldo.
struct CredJob {
    const void* P;
    int64_t ldp;
    const void* Q;
    int64_t ldq;
    int64_t M, N;
    void* out;
    int64_t ldo;
};

// `count` weight gradients over the same ntok tokens in one launch, each
// 128 x 128 tile on a cluster of S CTAs that split its tokens and reduce the
// partials on chip (splitk_cluster.cuh); bf16 store or fp32 accumulate.
cola_status_t run_cluster_wgrad(int count, const CredJob* jobs, int64_t ntok, int S, bool accumulate_f32,
                                unsigned int* status, cudaStream_t st)
{
    CredBatch b;
    std::memset(&b, 0, sizeof b);
    const int kb = static_cast<int>((ntok + BK - 1) / BK);
    b.count = count;
    b.S = S;
    b.kps = (kb + S - 1) / S;
    b.op = accumulate_f32 ? CRED_ACC : CRED_STORE;
    b.status = status;
    int64_t mnk[MAX_GROUP][3];
    double flops = 0.0;
    int tiles = 0;
    for (int j = 0; j < count; ++j) {
        const CredJob& J = jobs[j];
        CredProblem& P = b.prob[j];
        COLA_MAP(map_mnmajor(&P.map_a, J.P, J.M, ntok, J.ldp));
        COLA_MAP(map_mnmajor(&P.map_b, J.Q, J.N, ntok, J.ldq));
        P.M = static_cast<int>(J.M);
        P.N = static_cast<int>(J.N);
        P.k_blocks = kb;
        P.m_tiles = static_cast<int>((J.M + BM - 1) / BM);
        P.n_tiles = static_cast<int>((J.N + CBN - 1) / CBN);
        P.tile_begin = tiles;
        tiles += P.m_tiles * P.n_tiles;
        P.out = J.out;
        P.ldo = J.ldo;
        mnk[j][0] = J.M;
        mnk[j][1] = J.N;
        mnk[j][2] = ntok;
        flops += 2.0 * J.M * J.N * ntok;
    }
    b.tiles = tiles;
    return launched(traced(COLA_KERNEL_WGRAD, count, mnk, S, TRACE_CLUSTER, st,
                           [&] { return launch_splitk_cluster(b, flops < 64e9, st); }));
}

// A reduce launch after a split weight-gradient launch, in k-block steps of
// the busiest CTA (a few microseconds), for the comparison below.
constexpr double REDUCE_LAUNCH_KB = 16.0;

// The cluster split of a weight-gradient group (128 x 128 tiles, at most 8
// splits, one wave of clusters): > 1 when it applies -- each CTA walks at
// most CLUSTER_MAX_KPS k-blocks -- and its k-blocks per CTA undercut the
// planned schedule with its reduce launch.  Its 4-stage, one-tile-per-CTA
// form is made for short token walks: at 65536 tokens (the LLaMA-60M block,
// 128-171 k-blocks per CTA) it ran the weight gradients 60 -> 93 us.
constexpr int CLUSTER_MAX_KPS = 16;

int wgrad_cluster_splits(const WgradPlan& w, int64_t ntok, int accumulate_f32, int sms)
{
    if (!g_cluster_splitk.load(std::memory_order_relaxed)) return 1;
    int tiles = 0;
    for (int j = 0; j < w.count; ++j)
        tiles += static_cast<int>(((w.p[j].M + BM - 1) / BM) * ((w.p[j].N + CBN - 1) / CBN));
    const int kb = static_cast<int>((ntok + BK - 1) / BK);
    const int S = cluster_splits(tiles, kb, sms);
    if (S < 2 || (kb + S - 1) / S > CLUSTER_MAX_KPS) return 1;
    double planned = w.cost + REDUCE_LAUNCH_KB;
    if (!accumulate_f32) {
        const TailPlan tp = wgrad_tail_plan(w, ntok, sms);
        if (tail_wins(w, tp)) planned = tp.cost + (tp.pieces > 1 ? REDUCE_LAUNCH_KB : 0.0);
    }
    return (kb + S - 1) / S <= planned ? S : 1;
}

// F1: Z = X A^T, H = sigma(Z)  (N = r, or 3r for the fused q/k/v factors;
// Z / H pitch ldz)
cola_status_t run_f1(const Shape& s, int sigma, int64_t N, const void* X, const void* A, void* Z, void* H,
                     int64_t ldz, float* part, size_t part_bytes, unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn_for(s.n, N, s.d_in);
    const int ms = choose_msub(s.n, N, s.d_in, bn);
    GemmProblem pr;
    std::memset(&pr, 0, sizeof pr);
    pr.p = base_params(s.n, N, s.d_in, bn, ms);
    COLA_MAP(map_kmajor(&pr.map_a, X, s.d_in, s.n, s.ld_x, a_box_rows(ms)));
    COLA_MAP(map_kmajor(&pr.map_b, A, s.d_in, N, s.ld_a, b_box_rows(bn, ms)));
    const int S = ms == 1 ? small_launch_splits(pr.p.m_tiles * pr.p.n_tiles, pr.p.k_blocks, sms) : 1;
    if (S > 1) {
        // a small launch: K split across CTAs into fp32 partials, then the
        // reduce applies the Z/H epilogue (Z = bf16(sum), H = bf16(sigma(Z)))
        set_splits(pr.p, S);
        const int64_t slab = partial_elems(pr.p, bn, 1);
        if (static_cast<size_t>(pr.p.splits * slab) * 4 > part_bytes) return COLA_ERR_WORKSPACE;
        pr.map_d = pr.map_d2 = pr.map_z = pr.map_a;
        pr.p.D = part;
        pr.p.ldd = static_cast<long long>(pr.p.n_tiles) * bn;
        pr.p.part_stride = slab;
        pr.p.status = status;
        const int64_t mnk[1][3] = {{s.n, N, s.d_in}};
        COLA_TRY((run_batch<false, false, EPI_F32>(COLA_KERNEL_FWD_ZH, bn, 1, &pr, mnk, 1, 2, sms, st)));
        ReduceBatch rb;
        std::memset(&rb, 0, sizeof rb);
        rb.count = 1;
        rb.splits = pr.p.splits;
        rb.zh = 1;
        rb.sigma = sigma;
        ReduceJob& rj = rb.job[0];
        rj.part = part;
        rj.part_stride = slab;
        rj.ldp = pr.p.n_tiles * bn;
        rj.M = static_cast<int>(s.n);
        rj.N = static_cast<int>(N);
        rj.out = Z;
        rj.out2 = H;
        rj.ldo = ldz;
        const int64_t rmnk[1][3] = {{s.n, N, pr.p.splits}};
        return launched(traced(COLA_KERNEL_REDUCE, 1, rmnk, pr.p.splits, Z ? 1 : 0, st,
                               [&] { return launch_splitk_reduce(rb, st); }));
    }
    // Z == nullptr (inference): the epilogue stores H alone, through map_d
    COLA_MAP(map_box32(&pr.map_d, Z ? Z : H, N, s.n, ldz));
    pr.map_d2 = pr.map_d;
    if (Z && H) COLA_MAP(map_box32(&pr.map_d2, H, N, s.n, ldz));
    pr.map_z = pr.map_d;
    pr.p.has_d2 = Z && H;
    pr.p.h_only = Z == nullptr;
    pr.p.sigma = sigma;
    pr.p.status = status;
    const int64_t mnk[1][3] = {{s.n, N, s.d_in}};
    return run_batch<false, false, EPI_ZH>(COLA_KERNEL_FWD_ZH, bn, ms, &pr, mnk, 1, Z && H, sms, st);
}

}  // namespace

cudaError_t launch_fused_layer(const FusedParams& p, int r, bool bwd, int grid, bool pdl, cudaStream_t stream);

namespace {

// Whether cola_fwd / cola_bwd run a layer's two products as one fused kernel
// where that form applies (cola_set_fused_forward / cola_set_fused_backward).
std::atomic<int> g_fused_fwd{1};
std::atomic<int> g_fused_bwd{1};

// The single-kernel forward applies to one layer with r = 64 or 128 whose
// two GEMMs are HBM-bound (neither is compute-heavy), with at most one
// 128-row tile per SM, and not split over K (small launches keep the
// split-K forward).  Measured at 2048 tokens: -10 to -13 % against the two
// GEMMs; at 65536 tokens it was 5-13 % slower, so larger launches keep them.
bool fused_fwd_applies(const Shape& s, int sms)
{
    if (!g_fused_fwd.load(std::memory_order_relaxed) || (s.r != 64 && s.r != 128)) return false;
    if ((s.n + BM - 1) / BM > sms) return false;
    if (heavy_gemm(s.n, s.r, s.d_in) || heavy_gemm(s.n, s.d_out, s.r)) return false;
    GemmParams p1 = base_params(s.n, s.r, s.d_in, choose_bn_for(s.n, s.r, s.d_in), 1);
    if (small_launch_splits(p1.m_tiles * p1.n_tiles, p1.k_blocks, sms) > 1) return false;
    GemmParams p2 = base_params(s.n, s.d_out, s.r, choose_bn_for(s.n, s.d_out, s.r), 1);
    return small_launch_splits(p2.m_tiles * p2.n_tiles, p2.k_blocks, sms) == 1;
}

// The single-kernel dZ + dX applies on the same terms: r = 64 or 128, at
// most one 128-row tile per SM, neither GEMM compute-heavy (the backward's
// GEMMs are never split over K).
bool fused_bwd_applies(const Shape& s, int sms)
{
    if (!g_fused_bwd.load(std::memory_order_relaxed) || (s.r != 64 && s.r != 128)) return false;
    if ((s.n + BM - 1) / BM > sms) return false;
    return !heavy_gemm(s.n, s.r, s.d_out) && !heavy_gemm(s.n, s.d_in, s.r);
}

// Work items of a fused pass: the output blocks of a tile shared by up to
// sms / m_tiles items, so that the launch fills the SMs.
void fused_items(FusedParams& p, int sms)
{
    int groups = sms / (p.m_tiles > 0 ? p.m_tiles : 1);
    groups = std::max(1, std::min(groups, p.n_blocks));
    p.blocks_per_group = (p.n_blocks + groups - 1) / groups;
    p.out_groups = (p.n_blocks + p.blocks_per_group - 1) / p.blocks_per_group;
}

// F1 + F2 in one kernel: Z = X A^T, H = sigma(Z) kept on chip, Y = H B^T;
// Z and H stored when not null.
cola_status_t run_fused_fwd(const Shape& s, int sigma, const void* X, const void* A, const void* B, void* Y, void* Z,
                            void* H, unsigned int* status, int sms, cudaStream_t st)
{
    FusedParams p;
    std::memset(&p, 0, sizeof p);
    COLA_MAP(map_kmajor(&p.map_in, X, s.d_in, s.n, s.ld_x, BM));
    COLA_MAP(map_kmajor(&p.map_w1, A, s.d_in, s.r, s.ld_a, static_cast<int>(s.r)));
    COLA_MAP(map_kmajor(&p.map_w2, B, s.r, s.d_out, s.r, FBN));
    COLA_MAP(map_box32(&p.map_out, Y, s.d_out, s.n, s.ld_y));
    p.map_zin = p.map_s1 = p.map_s2 = p.map_out;
    if (Z) COLA_MAP(map_box32(&p.map_s1, Z, s.r, s.n, s.r));
    if (H) COLA_MAP(map_box32(&p.map_s2, H, s.r, s.n, s.r));
    p.n = static_cast<int>(s.n);
    p.n_out = static_cast<int>(s.d_out);
    p.kb1 = static_cast<int>((s.d_in + BK - 1) / BK);
    p.m_tiles = static_cast<int>((s.n + BM - 1) / BM);
    p.n_blocks = static_cast<int>((s.d_out + FBN - 1) / FBN);
    fused_items(p, sms);
    p.store_s1 = Z != nullptr;
    p.store_s2 = H != nullptr;
    p.sigma = sigma;
    p.out_ptr = static_cast<__nv_bfloat16*>(Y);
    p.out_ld = s.ld_y;
    p.status = status;
    const int items = p.m_tiles * p.out_groups;
    const int grid = items < sms ? items : sms;
    const double flops = 2.0 * s.n * s.r * (s.d_in + s.d_out);
    const int64_t mnk[2][3] = {{s.n, s.r, s.d_in}, {s.n, s.d_out, s.r}};
    const int flags = (H ? 1 : 0) | (Z ? TRACE_Z : 0);
    return launched(traced(COLA_KERNEL_FWD_FUSED, 2, mnk, 1, flags, st,
                           [&] { return launch_fused_layer(p, static_cast<int>(s.r), false, grid, flops < 64e9, st); }));
}

// B1 + B4 in one kernel: dZ = (dY B) * sigma'(Z) kept on chip (and stored
// to dZ, pitch r), dX = dZ A; under CoLA-M H = sigma(Z) stored to Hrec
// (pitch r) for the weight gradient of B.
cola_status_t run_fused_bwd(const Shape& s, int sigma, const void* dY, const void* B, const void* Z, const void* A,
                            void* dX, void* dZ, void* Hrec, unsigned int* status, int sms, cudaStream_t st)
{
    FusedParams p;
    std::memset(&p, 0, sizeof p);
    COLA_MAP(map_kmajor(&p.map_in, dY, s.d_out, s.n, s.ld_y, BM));
    COLA_MAP(map_mnmajor(&p.map_w1, B, s.r, s.d_out, s.r));
    COLA_MAP(map_mnmajor(&p.map_w2, A, s.d_in, s.r, s.ld_a));
    COLA_MAP(map_kmajor(&p.map_zin, Z, s.r, s.n, s.r, BM));
    COLA_MAP(map_box32(&p.map_s1, dZ, s.r, s.n, s.r));
    p.map_s2 = p.map_s1;
    if (Hrec) COLA_MAP(map_box32(&p.map_s2, Hrec, s.r, s.n, s.r));
    COLA_MAP(map_box32(&p.map_out, dX, s.d_in, s.n, s.ld_x));
    p.n = static_cast<int>(s.n);
    p.n_out = static_cast<int>(s.d_in);
    p.kb1 = static_cast<int>((s.d_out + BK - 1) / BK);
    p.m_tiles = static_cast<int>((s.n + BM - 1) / BM);
    p.n_blocks = static_cast<int>((s.d_in + FBN - 1) / FBN);
    fused_items(p, sms);
    p.store_s1 = 1;
    p.store_s2 = Hrec != nullptr;
    p.sigma = sigma;
    p.out_ptr = static_cast<__nv_bfloat16*>(dX);
    p.out_ld = s.ld_x;
    p.status = status;
    const int items = p.m_tiles * p.out_groups;
    const int grid = items < sms ? items : sms;
    const double flops = 2.0 * s.n * s.r * (s.d_out + s.d_in);
    const int64_t mnk[2][3] = {{s.n, s.r, s.d_out}, {s.n, s.d_in, s.r}};
    const int flags = Hrec ? 1 : 0;
    return launched(traced(COLA_KERNEL_BWD_FUSED, 2, mnk, 1, flags, st,
                           [&] { return launch_fused_layer(p, static_cast<int>(s.r), true, grid, flops < 64e9, st); }));
}

// F2: Y_j = H_j B_j^T for `count` projections of one shape (H_j [n x r] with
// pitch ldh; Y_j pitch ld_y), one launch
cola_status_t run_f2(const Shape& s, int count, const void* const* H, int64_t ldh, const void* const* B,
                     void* const* Y, float* part, size_t part_bytes, unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn_for(s.n, s.d_out, s.r);
    const int ms = choose_msub(s.n, s.d_out, s.r, bn);
    GemmProblem pr[MAX_GROUP];
    int64_t mnk[MAX_GROUP][3];
    std::memset(pr, 0, sizeof pr);
    {
        const GemmParams p0 = base_params(s.n, s.d_out, s.r, bn, ms);
        const int S = ms == 1 ? small_launch_splits(count * p0.m_tiles * p0.n_tiles, p0.k_blocks, sms) : 1;
        if (S > 1) {
            // a small launch: K split into fp32 partials, reduced into bf16 Y_j
            ReduceBatch rb;
            std::memset(&rb, 0, sizeof rb);
            int64_t rmnk[MAX_GROUP][3];
            float* slab_base = part;
            for (int j = 0; j < count; ++j) {
                pr[j].p = p0;
                set_splits(pr[j].p, S);
                const int64_t slab = partial_elems(pr[j].p, bn, 1);
                if (static_cast<size_t>((slab_base - part) + pr[j].p.splits * slab) * 4 > part_bytes)
                    return COLA_ERR_WORKSPACE;
                COLA_MAP(map_kmajor(&pr[j].map_a, H[j], s.r, s.n, ldh, a_box_rows(1)));
                COLA_MAP(map_kmajor(&pr[j].map_b, B[j], s.r, s.d_out, s.r, b_box_rows(bn, 1)));
                pr[j].map_d = pr[j].map_d2 = pr[j].map_z = pr[j].map_a;
                pr[j].p.D = slab_base;
                pr[j].p.ldd = static_cast<long long>(pr[j].p.n_tiles) * bn;
                pr[j].p.part_stride = slab;
                pr[j].p.status = status;
                mnk[j][0] = s.n;
                mnk[j][1] = s.d_out;
                mnk[j][2] = s.r;
                ReduceJob& rj = rb.job[j];
                rj.part = slab_base;
                rj.part_stride = slab;
                rj.ldp = pr[j].p.n_tiles * bn;
                rj.M = static_cast<int>(s.n);
                rj.N = static_cast<int>(s.d_out);
                rj.out = Y[j];
                rj.ldo = s.ld_y;
                rmnk[j][0] = s.n;
                rmnk[j][1] = s.d_out;
                rmnk[j][2] = pr[j].p.splits;
                slab_base += pr[j].p.splits * slab;
            }
            COLA_TRY((run_batch<false, false, EPI_F32>(COLA_KERNEL_FWD_Y, bn, 1, pr, mnk, count, 2, sms, st)));
            rb.count = count;
            rb.splits = pr[0].p.splits;
            return launched(traced(COLA_KERNEL_REDUCE, count, rmnk, pr[0].p.splits, 0, st,
                                   [&] { return launch_splitk_reduce(rb, st); }));
        }
    }
    for (int j = 0; j < count; ++j) {
        pr[j].p = base_params(s.n, s.d_out, s.r, bn, ms);
        COLA_MAP(map_kmajor(&pr[j].map_a, H[j], s.r, s.n, ldh, a_box_rows(ms)));
        COLA_MAP(map_kmajor(&pr[j].map_b, B[j], s.r, s.d_out, s.r, b_box_rows(bn, ms)));
        COLA_MAP(map_box32(&pr[j].map_d, Y[j], s.d_out, s.n, s.ld_y));
        pr[j].map_d2 = pr[j].map_z = pr[j].map_d;
        pr[j].p.d_ptr = static_cast<__nv_bfloat16*>(Y[j]);
        pr[j].p.d_ld = s.ld_y;
        pr[j].p.status = status;
        mnk[j][0] = s.n;
        mnk[j][1] = s.d_out;
        mnk[j][2] = s.r;
    }
    return run_batch<false, false, EPI_STORE>(COLA_KERNEL_FWD_Y, bn, ms, pr, mnk, count, 0, sms, st);
}

// B1: dZ_j = (dY_j B_j) * sigma'(Z_j) for `count` projections (Z_j, dZ_j, H_j
// column blocks of pitch ldz); H_j = sigma(Z_j) too when Hout != null (CoLA-M)
cola_status_t run_b1(const Shape& s, int sigma, int count, const void* const* dY, const void* const* B,
                     const void* const* Z, int64_t ldz, void* const* dZ, void* const* Hout, unsigned int* status,
                     int sms, cudaStream_t st)
{
    const int bn = choose_bn_for(s.n, s.r, s.d_out);
    const int ms = choose_msub(s.n, s.r, s.d_out, bn);
    GemmProblem pr[MAX_GROUP];
    int64_t mnk[MAX_GROUP][3];
    std::memset(pr, 0, sizeof pr);
    for (int j = 0; j < count; ++j) {
        pr[j].p = base_params(s.n, s.r, s.d_out, bn, ms);
        COLA_MAP(map_kmajor(&pr[j].map_a, dY[j], s.d_out, s.n, s.ld_y, a_box_rows(ms)));
        COLA_MAP(map_mnmajor(&pr[j].map_b, B[j], s.r, s.d_out, s.r));
        COLA_MAP(map_box32(&pr[j].map_d, dZ[j], s.r, s.n, ldz));
        COLA_MAP(map_box32(&pr[j].map_z, Z[j], s.r, s.n, ldz));
        pr[j].map_d2 = pr[j].map_d;
        if (Hout) COLA_MAP(map_box32(&pr[j].map_d2, Hout[j], s.r, s.n, ldz));
        pr[j].p.has_d2 = Hout != nullptr;
        pr[j].p.sigma = sigma;
        pr[j].p.status = status;
        mnk[j][0] = s.n;
        mnk[j][1] = s.r;
        mnk[j][2] = s.d_out;
    }
    if (Hout) return run_batch<false, true, EPI_DSIGMA_H>(COLA_KERNEL_BWD_DZ, bn, ms, pr, mnk, count, 1, sms, st);
    return run_batch<false, true, EPI_DSIGMA>(COLA_KERNEL_BWD_DZ, bn, ms, pr, mnk, count, 0, sms, st);
}

// Weight gradients of one backward call, in one launch: D_j[M_j x N_j] =
// sum_t P_j[t, m] Q_j[t, n] over the n tokens, both operands token-major
// (MN-major).  bf16 gradients run with a split tail (run_wgrad_tail) when
// the planner's cost model prefers it; otherwise, and for fp32 gradients
// accumulated into (D += ...), the token range of every tile is split
// uniformly into fp32 partial slabs (laid out one gradient after another)
// that the reduce adds, in a fixed order, into (onto) D.
struct WgradJob {
    const void* P;
    int64_t ldp;
    const void* Q;
    int64_t ldq;
    void* out;
    int64_t ldo;
};

cola_status_t run_wgrad_tail(const WgradPlan& w, int64_t ntok, const WgradJob* jobs, float* part, size_t part_bytes,
                           unsigned int* status, int sms, cudaStream_t st);

cola_status_t run_wgrad(const WgradPlan& w, int64_t ntok, const WgradJob* jobs, int accumulate_f32, float* part,
                        size_t part_bytes, unsigned int* status, int sms, cudaStream_t st)
{
    {
        // a small launch: the token splits reduced inside clusters, when one
        // wave of clusters costs less than the planned schedule with its
        // reduce launch (counted as REDUCE_LAUNCH_KB k-block steps)
        const int Sc = wgrad_cluster_splits(w, ntok, accumulate_f32, sms);
        if (Sc > 1) {
            CredJob J[MAX_GROUP];
            for (int j = 0; j < w.count; ++j)
                J[j] = CredJob{jobs[j].P, jobs[j].ldp, jobs[j].Q, jobs[j].ldq, w.p[j].M, w.p[j].N, jobs[j].out, jobs[j].ldo};
            return run_cluster_wgrad(w.count, J, ntok, Sc, accumulate_f32 != 0, status, st);
        }
    }
    if (!accumulate_f32 && tail_wins(w, wgrad_tail_plan(w, ntok, sms)))
        return run_wgrad_tail(w, ntok, jobs, part, part_bytes, status, sms, st);
    if (static_cast<size_t>(w.part_elems) * 4 > part_bytes) return COLA_ERR_WORKSPACE;
    GemmProblem pr[MAX_GROUP];
    int64_t mnk[MAX_GROUP][3];
    std::memset(pr, 0, sizeof pr);
    ReduceBatch rb;
    std::memset(&rb, 0, sizeof rb);
    float* slab_base = part;
    for (int j = 0; j < w.count; ++j) {
        const GemmParams& pj = w.p[j];
        pr[j].p = pj;
        COLA_MAP(map_mnmajor(&pr[j].map_a, jobs[j].P, pj.M, ntok, jobs[j].ldp));
        COLA_MAP(map_mnmajor(&pr[j].map_b, jobs[j].Q, pj.N, ntok, jobs[j].ldq));
        pr[j].p.status = status;
        pr[j].map_d = pr[j].map_d2 = pr[j].map_z = pr[j].map_a;
        pr[j].p.D = slab_base;
        pr[j].p.ldd = static_cast<long long>(pj.n_tiles) * w.bn;
        pr[j].p.part_stride = w.slab[j];
        ReduceJob& rj = rb.job[j];
        rj.part = slab_base;
        rj.part_stride = w.slab[j];
        rj.ldp = pj.n_tiles * w.bn;
        rj.M = pj.M;
        rj.N = pj.N;
        rj.out = jobs[j].out;
        rj.ldo = jobs[j].ldo;
        slab_base += static_cast<int64_t>(pj.splits) * w.slab[j];
        mnk[j][0] = pj.M;
        mnk[j][1] = pj.N;
        mnk[j][2] = ntok;
    }
    COLA_TRY((run_batch<true, true, EPI_F32>(COLA_KERNEL_WGRAD, w.bn, w.msub, pr, mnk, w.count, 0, sms, st)));
    rb.count = w.count;
    rb.splits = w.splits;
    rb.accumulate_f32 = accumulate_f32;
    int64_t rmnk[MAX_GROUP][3];
    for (int j = 0; j < w.count; ++j) {
        rmnk[j][0] = w.p[j].M;
        rmnk[j][1] = w.p[j].N;
        rmnk[j][2] = w.splits;
    }
    return launched(traced(COLA_KERNEL_REDUCE, w.count, rmnk, w.splits, 0, st,
                           [&] { return launch_splitk_reduce(rb, st); }));
}

// bf16 weight gradients with a split tail: the whole tiles are stored
// straight from the GEMM epilogue; the pieces of the split tail tiles are
// summed by the tail reduce (no reduce when the tail is not split).
cola_status_t run_wgrad_tail(const WgradPlan& w, int64_t ntok, const WgradJob* jobs, float* part, size_t part_bytes,
                           unsigned int* status, int sms, cudaStream_t st)
{
    const TailPlan tp = wgrad_tail_plan(w, ntok, sms);
    if (static_cast<size_t>(tp.part_elems) * 4 > part_bytes) return COLA_ERR_WORKSPACE;
    GemmProblem pr[MAX_GROUP];
    int64_t mnk[MAX_GROUP][3];
    std::memset(pr, 0, sizeof pr);
    TailReduce rd;
    std::memset(&rd, 0, sizeof rd);
    for (int j = 0; j < w.count; ++j) {
        pr[j].p = base_params(w.p[j].M, w.p[j].N, ntok, w.bn, w.msub);
        pr[j].p.n_major = w.p[j].n_major;
        const GemmParams& pj = pr[j].p;
        COLA_MAP(map_mnmajor(&pr[j].map_a, jobs[j].P, pj.M, ntok, jobs[j].ldp));
        COLA_MAP(map_mnmajor(&pr[j].map_b, jobs[j].Q, pj.N, ntok, jobs[j].ldq));
        COLA_MAP(map_box32(&pr[j].map_d, jobs[j].out, pj.N, pj.M, jobs[j].ldo));
        pr[j].map_d2 = pr[j].map_z = pr[j].map_d;
        pr[j].p.d_ptr = static_cast<__nv_bfloat16*>(jobs[j].out);
        pr[j].p.d_ld = jobs[j].ldo;
        pr[j].p.status = status;
        mnk[j][0] = pj.M;
        mnk[j][1] = pj.N;
        mnk[j][2] = ntok;
        rd.out[j] = jobs[j].out;
        rd.ldo[j] = jobs[j].ldo;
        rd.M[j] = pj.M;
        rd.N[j] = pj.N;
    }
    COLA_TRY((run_batch<true, true, EPI_TAIL>(COLA_KERNEL_WGRAD, w.bn, w.msub, pr, mnk, w.count, 0, sms, st, &tp,
                                             part)));
    if (tp.ntiles == 0) return COLA_OK;
    rd.part = part;
    rd.tile_rows = tile_rows(w.msub);
    rd.tile_cols = w.bn;
    rd.ntiles = tp.ntiles;
    for (int t = 0; t < tp.ntiles; ++t) rd.tile[t] = tp.tile[t];
    const int64_t rmnk[1][3] = {{static_cast<int64_t>(tp.ntiles) * rd.tile_rows, rd.tile_cols, tp.pieces}};
    return launched(traced(COLA_KERNEL_REDUCE, 1, rmnk, tp.pieces, TRACE_TAIL, st,
                           [&] { return launch_tail_reduce(rd, sms, st); }));
}

// Gated MLP forward GEMM: per 128-column tile of M = Y_gate * Y_up (pitch
// ld_y), one K walk over [H_gate H_up] (H_cat, pitch ldh) whose gate half
// accumulates H_gate B_gate^T and whose up half H_up B_up^T, in two
// accumulators; Y_gate, Y_up are stored too when not null (training).
// Compute-heavy launches with r >= 512 run on CTA pairs.
cola_status_t run_glu(const Shape& s, const void* H_cat, int64_t ldh, const void* Bg, const void* Bu, void* M,
                      void* Yg, void* Yu, unsigned int* status, int sms, cudaStream_t st)
{
    const int64_t K2 = 2 * s.r;
    const bool pair = heavy_gemm(s.n, s.d_out, K2) && s.r >= 512;
    const int msub = pair ? TILE_PAIR : 1;
    // 256-column pair tiles hold one tile in TMEM, so the next tile's up half
    // waits for this tile's stores: worth it when the epilogue stores M alone
    // or a half runs long (r >= 1024).  Measured: 7B inference GLU 355 -> 230
    // us, 7B training -3 % per block; 1B training 912 -> 1110 us, which keeps
    // the double-buffered 128-column pair tiles.
    const int bn = pair && (Yg == nullptr || s.r >= 1024) ? 256 : 128;
    GemmBatch b;
    std::memset(&b, 0, sizeof b);
    b.count = 1;
    GemmProblem& pr = b.prob[0];
    pr.p = base_params(s.n, s.d_out, K2, bn, msub);
    pr.p.glu_half = static_cast<int>(s.r / BK);
    COLA_MAP(map_kmajor(&pr.map_a, H_cat, K2, s.n, ldh, a_box_rows(msub)));
    COLA_MAP(map_kmajor(&pr.map_b, Bg, s.r, s.d_out, s.r, b_box_rows(bn, msub)));
    COLA_MAP(map_kmajor(&pr.map_b2, Bu, s.r, s.d_out, s.r, b_box_rows(bn, msub)));
    COLA_MAP(map_box32(&pr.map_d, M, s.d_out, s.n, s.ld_y));
    pr.map_d2 = pr.map_d3 = pr.map_z = pr.map_d;
    if (Yg) {
        COLA_MAP(map_box32(&pr.map_d2, Yg, s.d_out, s.n, s.ld_y));
        COLA_MAP(map_box32(&pr.map_d3, Yu, s.d_out, s.n, s.ld_y));
    }
    pr.p.has_d2 = Yg != nullptr;
    pr.p.d_ptr = static_cast<__nv_bfloat16*>(M);
    pr.p.d2_ptr = static_cast<__nv_bfloat16*>(Yg);
    pr.p.d3_ptr = static_cast<__nv_bfloat16*>(Yu);
    pr.p.d_ld = s.ld_y;
    pr.p.status = status;
    const int64_t mnk[1][3] = {{s.n, s.d_out, K2}};
    const int flags = (Yg ? 1 : 0) | (pair ? TRACE_PAIR : 0);
    return launched(traced(COLA_KERNEL_FWD_GLU, 1, mnk, 1, flags, st, [&] { return dispatch_glu(bn, pair, b, sms, st); }));
}

// The down layer's input gradient when its input is M = Y_gate * Y_up: the
// dX GEMM dM = dZ A (dZ [n x K] pitch ldz) whose epilogue stores
// dY_gate = bf16(dM) * Y_up and dY_up = bf16(dM) * Y_gate (all pitch ld_x).
cola_status_t run_b4_glu(const Shape& s, int64_t K, const void* dZ, int64_t ldz, const void* A, const void* Yg,
                         const void* Yu, void* dYg, void* dYu, unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn_for(s.n, s.d_in, K);
    const int ms = choose_msub(s.n, s.d_in, K, bn);
    GemmProblem pr;
    std::memset(&pr, 0, sizeof pr);
    pr.p = base_params(s.n, s.d_in, K, bn, ms);
    COLA_MAP(map_kmajor(&pr.map_a, dZ, K, s.n, ldz, a_box_rows(ms)));
    COLA_MAP(map_mnmajor(&pr.map_b, A, s.d_in, K, s.ld_a));
    COLA_MAP(map_box32(&pr.map_d, dYg, s.d_in, s.n, s.ld_x));
    COLA_MAP(map_box32(&pr.map_d2, dYu, s.d_in, s.n, s.ld_x));
    pr.map_z = pr.map_d3 = pr.map_b2 = pr.map_d;
    pr.p.d_ptr = static_cast<__nv_bfloat16*>(dYg);
    pr.p.d2_ptr = static_cast<__nv_bfloat16*>(dYu);
    pr.p.d_ld = s.ld_x;
    pr.p.yg_ptr = static_cast<const __nv_bfloat16*>(Yg);
    pr.p.yu_ptr = static_cast<const __nv_bfloat16*>(Yu);
    pr.p.status = status;
    const int64_t mnk[1][3] = {{s.n, s.d_in, K}};
    return run_batch<false, true, EPI_GLU_BWD>(COLA_KERNEL_BWD_DX, bn, ms, &pr, mnk, 1, TRACE_GLU, sms, st);
}

// B4: dX = dZ A  (dZ [n x K] pitch ldz, A [K x d_in] pitch ld_a; K = r or 3r)
cola_status_t run_b4(const Shape& s, int64_t K, const void* dZ, int64_t ldz, const void* A, void* dX,
                     unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn_for(s.n, s.d_in, K);
    const int ms = choose_msub(s.n, s.d_in, K, bn);
    GemmProblem pr;
    std::memset(&pr, 0, sizeof pr);
    pr.p = base_params(s.n, s.d_in, K, bn, ms);
    COLA_MAP(map_kmajor(&pr.map_a, dZ, K, s.n, ldz, a_box_rows(ms)));
    COLA_MAP(map_mnmajor(&pr.map_b, A, s.d_in, K, s.ld_a));
    COLA_MAP(map_box32(&pr.map_d, dX, s.d_in, s.n, s.ld_x));
    pr.map_d2 = pr.map_z = pr.map_d;
    pr.p.d_ptr = static_cast<__nv_bfloat16*>(dX);
    pr.p.d_ld = s.ld_x;
    pr.p.status = status;
    const int64_t mnk[1][3] = {{s.n, s.d_in, K}};
    return run_batch<false, true, EPI_STORE>(COLA_KERNEL_BWD_DX, bn, ms, &pr, mnk, 1, 0, sms, st);
}

}  // namespace
}  // namespace cola

using namespace cola;

extern "C" {

cola_status_t cola_workspace_size(const cola_desc_t* desc, int32_t nproj, size_t* bytes)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (!bytes || nproj < 1 || nproj > 3) return COLA_ERR_INVALID;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    *bytes = ws_layout(*desc, nproj, sms).total;
    return COLA_OK;
}

cola_status_t cola_workspace_init(void* ws, void* stream)
{
    if (!ws) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    return launched(cudaMemsetAsync(ws, 0, WS_HEADER, static_cast<cudaStream_t>(stream)));
}

cola_status_t cola_fwd(const cola_desc_t* desc, const void* X, const void* A, const void* B, void* Y,
                       void* Z_save, void* H_save, void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    COLA_TRY(check_ptrs({X, A, B, Y}));
    COLA_TRY(check_saved(desc->mode, Z_save, H_save));
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 1, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    void* H = desc->mode != COLA_MODE_COLA ? static_cast<void*>(wsb(ws) + L.h_off) : H_save;
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    if (fused_fwd_applies(s, sms))
        return run_fused_fwd(s, desc->sigma, X, A, B, Y, Z_save, H_save, status, sms, st);
    COLA_TRY(run_f1(s, desc->sigma, s.r, X, A, Z_save, H, s.r, part, part_bytes, status, sms, st));
    const void* Hs[1] = {H};
    const void* Bs[1] = {B};
    void* Ys[1] = {Y};
    return run_f2(s, 1, Hs, s.r, Bs, Ys, part, part_bytes, status, sms, st);
}

}  // extern "C"

namespace cola {
namespace {

// The gated-MLP ends of the down layer's backward (cola_bwd_down_gated).
struct GluBwd {
    const void* Yg;
    const void* Yu;
    void* dYg;
    void* dYu;
};

cola_status_t bwd_single(const cola_desc_t* desc, const void* X, const void* A, const void* B, const void* dY,
                         const void* Z_save, const void* H_save, void* dX, void* dA, void* dB, void* ws,
                         size_t ws_bytes, void* stream, const GluBwd* glu)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (desc->mode == COLA_MODE_INFER) return COLA_ERR_INVALID;
    COLA_TRY(check_ptrs({X, A, B, dY, Z_save, dA, dB}));
    if (glu)
        COLA_TRY(check_ptrs({glu->Yg, glu->Yu, glu->dYg, glu->dYu}));
    else
        COLA_TRY(check_ptrs({dX}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_save != nullptr : H_save == nullptr) return COLA_ERR_INVALID;
    if (H_save && !aligned16(H_save)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 1, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    void* dZ = wsb(ws) + L.dz_off;
    void* Hrec = cola_m ? static_cast<void*>(wsb(ws) + L.h_off) : nullptr;
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;

    const void* dYs[1] = {dY};
    const void* Bs[1] = {B};
    const void* Zs[1] = {Z_save};
    void* dZs[1] = {dZ};
    void* Hs[1] = {Hrec};
    const void* Hsrc = cola_m ? Hrec : H_save;
    const WgradPlan w = wgrad_plan(*desc, 1, sms);
    const WgradJob jobs[2] = {{dY, s.ld_y, Hsrc, s.r, dB, s.r}, {dZ, s.r, X, s.ld_x, dA, s.ld_a}};
    if (!glu && fused_bwd_applies(s, sms)) {
        // dZ (and H) with dX in one kernel, then the weight gradients
        COLA_TRY(run_fused_bwd(s, desc->sigma, dY, B, Z_save, A, dX, dZ, Hrec, status, sms, st));
        return run_wgrad(w, s.n, jobs, desc->wgrad_fp32, part, part_bytes, status, sms, st);
    }
    COLA_TRY(run_b1(s, desc->sigma, 1, dYs, Bs, Zs, s.r, dZs, cola_m ? Hs : nullptr, status, sms, st));
    COLA_TRY(run_wgrad(w, s.n, jobs, desc->wgrad_fp32, part, part_bytes, status, sms, st));
    if (glu) return run_b4_glu(s, s.r, dZ, s.r, A, glu->Yg, glu->Yu, glu->dYg, glu->dYu, status, sms, st);
    return run_b4(s, s.r, dZ, s.r, A, dX, status, sms, st);
}

}  // namespace
}  // namespace cola

extern "C" {

cola_status_t cola_bwd(const cola_desc_t* desc, const void* X, const void* A, const void* B, const void* dY,
                       const void* Z_save, const void* H_save, void* dX, void* dA, void* dB, void* ws,
                       size_t ws_bytes, void* stream)
{
    return bwd_single(desc, X, A, B, dY, Z_save, H_save, dX, dA, dB, ws, ws_bytes, stream, nullptr);
}

cola_status_t cola_bwd_down_gated(const cola_desc_t* desc, const void* M, const void* A, const void* B,
                                  const void* dY, const void* Z_save, const void* H_save, const void* Y_gate,
                                  const void* Y_up, void* dY_gate, void* dY_up, void* dA, void* dB, void* ws,
                                  size_t ws_bytes, void* stream)
{
    const GluBwd glu{Y_gate, Y_up, dY_gate, dY_up};
    return bwd_single(desc, M, A, B, dY, Z_save, H_save, nullptr, dA, dB, ws, ws_bytes, stream, &glu);
}

cola_status_t cola_fwd_gate_up(const cola_desc_t* desc, const void* X, const void* A_cat, const void* B_gate,
                               const void* B_up, void* M, void* Y_gate, void* Y_up, void* Z_cat, void* H_cat,
                               void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    COLA_TRY(check_ptrs({X, A_cat, B_gate, B_up, M}));
    COLA_TRY(check_saved(desc->mode, Z_cat, H_cat));
    const bool train = desc->mode != COLA_MODE_INFER;
    if ((Y_gate != nullptr) != train || (Y_up != nullptr) != train) return COLA_ERR_INVALID;
    if ((Y_gate && !aligned16(Y_gate)) || (Y_up && !aligned16(Y_up))) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 2, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = 2 * s.r;
    uint8_t* H = desc->mode != COLA_MODE_COLA ? wsb(ws) + L.h_off : static_cast<uint8_t*>(H_cat);
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    COLA_TRY(run_f1(s, desc->sigma, R, X, A_cat, Z_cat, H, R, part, part_bytes, status, sms, st));
    return run_glu(s, H, R, B_gate, B_up, M, Y_gate, Y_up, status, sms, st);
}

cola_status_t cola_fwd_shared_x(const cola_desc_t* desc, int32_t count, const void* X, const void* A_cat,
                                const void* const* B, void* const* Y, void* Z_cat, void* H_cat, void* ws,
                                size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (count < 2 || count > 3 || !B || !Y) return COLA_ERR_INVALID;
    COLA_TRY(check_ptrs({X, A_cat}));
    for (int j = 0; j < count; ++j) COLA_TRY(check_ptrs({B[j], Y[j]}));
    COLA_TRY(check_saved(desc->mode, Z_cat, H_cat));
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, count, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = count * s.r;
    const size_t slice = static_cast<size_t>(s.r) * 2;   // bytes between the projections' column blocks
    uint8_t* H = desc->mode != COLA_MODE_COLA ? wsb(ws) + L.h_off : static_cast<uint8_t*>(H_cat);
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    COLA_TRY(run_f1(s, desc->sigma, R, X, A_cat, Z_cat, H, R, part, part_bytes, status, sms, st));
    const void* Hs[3] = {H, H + slice, H + 2 * slice};
    return run_f2(s, count, Hs, R, B, Y, part, part_bytes, status, sms, st);
}

cola_status_t cola_bwd_shared_x(const cola_desc_t* desc, int32_t count, const void* X, const void* A_cat,
                                const void* const* B, const void* const* dY, const void* Z_cat, const void* H_cat,
                                void* dX, void* dA_cat, void* const* dB, void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (count < 2 || count > 3 || !B || !dY || !dB || desc->mode == COLA_MODE_INFER) return COLA_ERR_INVALID;
    COLA_TRY(check_ptrs({X, A_cat, Z_cat, dX, dA_cat}));
    for (int j = 0; j < count; ++j) COLA_TRY(check_ptrs({B[j], dY[j], dB[j]}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_cat != nullptr : H_cat == nullptr) return COLA_ERR_INVALID;
    if (H_cat && !aligned16(H_cat)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, count, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = count * s.r;
    const size_t slice = static_cast<size_t>(s.r) * 2;   // bytes between the projections' column blocks
    uint8_t* dZ = wsb(ws) + L.dz_off;
    uint8_t* Hrec = cola_m ? wsb(ws) + L.h_off : nullptr;
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    const uint8_t* Zb = static_cast<const uint8_t*>(Z_cat);
    const uint8_t* Hsrc = cola_m ? Hrec : static_cast<const uint8_t*>(H_cat);

    const void* Zs[3];
    void* dZs[3];
    void* Hr[3];
    WgradJob jobs[MAX_GROUP];
    for (int j = 0; j < count; ++j) {
        Zs[j] = Zb + j * slice;
        dZs[j] = dZ + j * slice;
        Hr[j] = Hrec ? Hrec + j * slice : nullptr;
        jobs[j] = {dY[j], s.ld_y, Hsrc + j * slice, R, dB[j], s.r};
    }
    jobs[count] = {dZ, R, X, s.ld_x, dA_cat, s.ld_a};
    COLA_TRY(run_b1(s, desc->sigma, count, dY, B, Zs, R, dZs, cola_m ? Hr : nullptr, status, sms, st));
    const WgradPlan w = wgrad_plan(*desc, count, sms);
    COLA_TRY(run_wgrad(w, s.n, jobs, desc->wgrad_fp32, part, part_bytes, status, sms, st));
    return run_b4(s, R, dZ, R, A_cat, dX, status, sms, st);
}

cola_status_t cola_fwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, void* Y_q, void* Y_k, void* Y_v, void* Z_qkv,
                                 void* H_qkv, void* ws, size_t ws_bytes, void* stream)
{
    const void* B[3] = {B_q, B_k, B_v};
    void* Y[3] = {Y_q, Y_k, Y_v};
    return cola_fwd_shared_x(desc, 3, X, A_qkv, B, Y, Z_qkv, H_qkv, ws, ws_bytes, stream);
}

cola_status_t cola_bwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, const void* dY_q, const void* dY_k,
                                 const void* dY_v, const void* Z_qkv, const void* H_qkv, void* dX, void* dA_qkv,
                                 void* dB_q, void* dB_k, void* dB_v, void* ws, size_t ws_bytes, void* stream)
{
    const void* B[3] = {B_q, B_k, B_v};
    const void* dY[3] = {dY_q, dY_k, dY_v};
    void* dB[3] = {dB_q, dB_k, dB_v};
    return cola_bwd_shared_x(desc, 3, X, A_qkv, B, dY, Z_qkv, H_qkv, dX, dA_qkv, dB, ws, ws_bytes, stream);
}

cola_status_t cola_recompute_up(const cola_desc_t* desc, int32_t count, const void* Z_cat, const void* const* B,
                                void* const* Y, void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (desc->mode != COLA_MODE_COLA_M || count < 1 || count > 3 || !B || !Y) return COLA_ERR_INVALID;
    COLA_TRY(check_ptrs({Z_cat}));
    for (int j = 0; j < count; ++j) COLA_TRY(check_ptrs({B[j], Y[j]}));
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, count, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = count * s.r;
    uint8_t* H = wsb(ws) + L.h_off;
    const int64_t mnk[1][3] = {{s.n, R, 0}};
    COLA_TRY(launched(traced(COLA_KERNEL_SIGMA, 1, mnk, 1, 0, st, [&] {
        return launch_sigma(Z_cat, H, static_cast<long long>(s.n) * R, desc->sigma, sms, st);
    })));
    const size_t slice = static_cast<size_t>(s.r) * 2;
    const void* Hs[3] = {H, H + slice, H + 2 * slice};
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    return run_f2(s, count, Hs, R, B, Y, part, L.total - L.part_off, status, sms, st);
}

static_assert(COLA_STATUS_PRODUCER_TIMEOUT == ST_TIMEOUT_PRODUCER && COLA_STATUS_MMA_TIMEOUT == ST_TIMEOUT_MMA &&
                  COLA_STATUS_EPILOGUE_TIMEOUT == ST_TIMEOUT_EPILOGUE && COLA_STATUS_DRAIN_TIMEOUT == ST_TIMEOUT_DRAIN,
              "status bits of the header and the kernels agree");

cola_status_t cola_selftest_wait_timeout(void* ws, size_t ws_bytes, void* stream)
{
    if (!ws) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    constexpr size_t tile_bytes = 128 * 128 * 2;
    if (ws_bytes < WS_HEADER + 3 * tile_bytes) return COLA_ERR_WORKSPACE;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    // one 128 x 128 x 64 GEMM whose operands and output lie in the workspace;
    // its producer issues no loads, so nothing is ever read or written there
    uint8_t* base = wsb(ws) + WS_HEADER;
    GemmProblem pr;
    std::memset(&pr, 0, sizeof pr);
    pr.p = base_params(128, 128, 64, 128, 1);
    COLA_MAP(map_kmajor(&pr.map_a, base, 64, 128, 64, BM));
    COLA_MAP(map_kmajor(&pr.map_b, base + tile_bytes, 64, 128, 64, 128));
    COLA_MAP(map_box32(&pr.map_d, base + 2 * tile_bytes, 128, 128, 128));
    pr.map_d2 = pr.map_z = pr.map_d;
    pr.p.d_ptr = reinterpret_cast<__nv_bfloat16*>(base + 2 * tile_bytes);
    pr.p.d_ld = 128;
    pr.p.status = ws_status(ws);
    pr.p.selftest = 1;
    const int64_t mnk[1][3] = {{128, 128, 64}};
    return run_batch<false, false, EPI_STORE>(COLA_KERNEL_FWD_Y, 128, 1, &pr, mnk, 1, 0, sms,
                                              static_cast<cudaStream_t>(stream));
}

cola_status_t cola_selftest_wait_timeout_pair(void* ws, size_t ws_bytes, int32_t variant, void* stream)
{
    if (!ws || (variant != 1 && variant != 2)) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    constexpr int64_t M = 256, N = 256, K = 512;   // one 256 x 256 pair tile, 8 k-blocks
    constexpr size_t a_bytes = M * K * 2, b_bytes = N * K * 2, d_bytes = M * N * 2;
    if (ws_bytes < WS_HEADER + a_bytes + b_bytes + d_bytes) return COLA_ERR_WORKSPACE;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    uint8_t* base = wsb(ws) + WS_HEADER;
    GemmProblem pr;
    std::memset(&pr, 0, sizeof pr);
    pr.p = base_params(M, N, K, 256, TILE_PAIR);
    COLA_MAP(map_kmajor(&pr.map_a, base, K, M, K, a_box_rows(TILE_PAIR)));
    COLA_MAP(map_kmajor(&pr.map_b, base + a_bytes, K, N, K, b_box_rows(256, TILE_PAIR)));
    COLA_MAP(map_box32(&pr.map_d, base + a_bytes + b_bytes, N, M, N));
    pr.map_d2 = pr.map_z = pr.map_d;
    pr.p.d_ptr = reinterpret_cast<__nv_bfloat16*>(base + a_bytes + b_bytes);
    pr.p.d_ld = N;
    pr.p.status = ws_status(ws);
    pr.p.selftest = variant;
    const int64_t mnk[1][3] = {{M, N, K}};
    return run_batch<false, false, EPI_STORE>(COLA_KERNEL_FWD_Y, 256, TILE_PAIR, &pr, mnk, 1, 0, sms,
                                              static_cast<cudaStream_t>(stream));
}

cola_status_t cola_selftest_wait_timeout_cluster(void* ws, size_t ws_bytes, void* stream)
{
    if (!ws) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    constexpr int64_t M = 128, N = 128, T = 512;   // one 128 x 128 gradient tile over 512 tokens
    constexpr size_t p_bytes = T * M * 2, q_bytes = T * N * 2;
    if (ws_bytes < WS_HEADER + p_bytes + q_bytes) return COLA_ERR_WORKSPACE;
    uint8_t* base = wsb(ws) + WS_HEADER;
    CredBatch b;
    std::memset(&b, 0, sizeof b);
    b.count = 1;
    b.tiles = 1;
    b.S = 2;
    b.kps = 4;
    b.op = CRED_STORE;
    b.status = ws_status(ws);
    b.selftest = 1;
    CredProblem& P = b.prob[0];
    COLA_MAP(map_mnmajor(&P.map_a, base, M, T, M));
    COLA_MAP(map_mnmajor(&P.map_b, base + p_bytes, N, T, N));
    P.M = static_cast<int>(M);
    P.N = static_cast<int>(N);
    P.k_blocks = static_cast<int>(T / BK);
    P.m_tiles = P.n_tiles = 1;
    // the owner that completes normally stores its band over the operand P
    // (already read by then); the CTA that gave up stores nothing
    P.out = base;
    P.ldo = N;
    const int64_t mnk[1][3] = {{M, N, T}};
    return launched(traced(COLA_KERNEL_WGRAD, 1, mnk, 2, TRACE_CLUSTER, static_cast<cudaStream_t>(stream),
                           [&] { return launch_splitk_cluster(b, false, static_cast<cudaStream_t>(stream)); }));
}

cola_status_t cola_check_status(void* ws, void* stream, uint32_t* code_out)
{
    if (!ws) return COLA_ERR_INVALID;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(st) != cudaSuccess) return COLA_ERR_LAUNCH;
    uint32_t code = 0;
    if (cudaMemcpy(&code, ws, sizeof code, cudaMemcpyDeviceToHost) != cudaSuccess) return COLA_ERR_LAUNCH;
    if (code_out) *code_out = code;
    if (code != 0) {
        if (cudaMemset(ws, 0, sizeof code) != cudaSuccess) return COLA_ERR_LAUNCH;
        return COLA_ERR_DEVICE_TIMEOUT;
    }
    return COLA_OK;
}

cola_status_t cola_set_fused_forward(int32_t enable)
{
    if (enable != 0 && enable != 1) return COLA_ERR_INVALID;
    g_fused_fwd.store(enable, std::memory_order_relaxed);
    return COLA_OK;
}

cola_status_t cola_set_fused_backward(int32_t enable)
{
    if (enable != 0 && enable != 1) return COLA_ERR_INVALID;
    g_fused_bwd.store(enable, std::memory_order_relaxed);
    return COLA_OK;
}

cola_status_t cola_set_cluster_splitk(int32_t enable)
{
    if (enable != 0 && enable != 1) return COLA_ERR_INVALID;
    g_cluster_splitk.store(enable, std::memory_order_relaxed);
    return COLA_OK;
}

cola_status_t cola_trace_attach(cola_trace_slot_t* slots, int32_t capacity, int32_t* count)
{
    if (!slots || !count || capacity < 0) return COLA_ERR_INVALID;
    for (int32_t i = 0; i < capacity; ++i)
        if (!slots[i].start || !slots[i].stop) return COLA_ERR_INVALID;
    g_trace.slots = slots;
    g_trace.capacity = capacity;
    g_trace.count = count;
    return COLA_OK;
}

cola_status_t cola_trace_detach(void)
{
    g_trace = TraceState{};
    return COLA_OK;
}

const char* cola_status_string(cola_status_t status)
{
    switch (status) {
    case COLA_OK: return "ok";
    case COLA_ERR_INVALID: return "invalid argument (null pointer, size, pitch or enum)";
    case COLA_ERR_ALIGN: return "misaligned pointer (16-byte; workspace 256-byte)";
    case COLA_ERR_UNSUPPORTED: return "unsupported shape or device (r % 64, extent, sm_103 required)";
    case COLA_ERR_WORKSPACE: return "workspace too small";
    case COLA_ERR_LAUNCH: return "CUDA launch or driver call failed";
    case COLA_ERR_DEVICE_TIMEOUT: return "a bounded device-side wait ran out";
    }
    return "unknown status";
}

}  // extern "C"
