// cola_abi.cu -- the extern "C" entry points of libcola.so (declared in
// include/cola.h): argument validation, workspace layout, TMA descriptors and
// the launch sequence of each pass of the CoLA layer.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <mutex>

#include "cola.h"
#include "gemm_launch.cuh"
#include "host_plan.cuh"

namespace cola {
namespace {

// ------------------------------------------------------------ device info
struct DevInfo {
    int ok = 0;      // 1: queried, 2: unsupported device
    int sms = 0;
};

DevInfo g_dev[64];
std::mutex g_mu;

cola_status_t device_info(int* sms)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return COLA_ERR_LAUNCH;
    DevInfo& d = g_dev[dev];
    if (d.ok == 0) {
        std::lock_guard<std::mutex> lock(g_mu);
        if (d.ok == 0) {
            int major = 0, minor = 0, n = 0;
            if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
                return COLA_ERR_LAUNCH;
            d.sms = n;
            d.ok = (major == 10 && minor == 3) ? 1 : 2;   // kernels are built for sm_103a only
        }
    }
    if (d.ok != 1) return COLA_ERR_UNSUPPORTED;
    *sms = d.sms;
    return COLA_OK;
}

// ------------------------------------------------------------ workspace
constexpr size_t WS_HEADER = 256;
constexpr size_t WS_ALIGN = 256;

size_t align_up(size_t v) { return (v + WS_ALIGN - 1) / WS_ALIGN * WS_ALIGN; }

struct WsLayout {
    size_t dz_off, h_off, part_off, total;
};

// dZ [n x R] bf16, H [n x R] bf16 (CoLA-M only), fp32 split-K partial slabs
// sized for the larger of the two weight-gradient GEMMs.
WsLayout ws_layout(const cola_desc_t& d, int fused, int sms)
{
    const int64_t R = fused ? 3 * d.r : d.r;
    WsLayout L;
    size_t off = WS_HEADER;
    L.dz_off = off;
    off += align_up(static_cast<size_t>(d.n) * R * 2);
    L.h_off = off;
    if (d.mode == COLA_MODE_COLA_M) off += align_up(static_cast<size_t>(d.n) * R * 2);
    L.part_off = off;
    const int bn_b = choose_bn(d.r);
    const int ms_b = choose_msub(d.d_out, d.r, d.n, bn_b);
    GemmParams pb = plan(d.d_out, d.r, d.n, bn_b, ms_b, sms, true);
    const int bn_a = choose_bn(d.d_in);
    const int ms_a = choose_msub(R, d.d_in, d.n, bn_a);
    GemmParams pa = plan(R, d.d_in, d.n, bn_a, ms_a, sms, true);
    const size_t part_b = static_cast<size_t>(pb.splits) * partial_elems(pb, bn_b, ms_b) * 4;
    const size_t part_a = static_cast<size_t>(pa.splits) * partial_elems(pa, bn_a, ms_a) * 4;
    off += align_up(part_b > part_a ? part_b : part_a);
    L.total = off;
    return L;
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
    if (d->mode != COLA_MODE_COLA && d->mode != COLA_MODE_COLA_M) return COLA_ERR_INVALID;
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

cola_status_t check_ws(const cola_desc_t& d, int fused, int sms, void* ws, size_t ws_bytes, WsLayout* L)
{
    if (!ws) return COLA_ERR_INVALID;
    if (reinterpret_cast<uintptr_t>(ws) & (WS_ALIGN - 1)) return COLA_ERR_ALIGN;
    *L = ws_layout(d, fused, sms);
    if (ws_bytes < L->total) return COLA_ERR_WORKSPACE;
    return COLA_OK;
}

inline cola_status_t launched(cudaError_t e) { return e == cudaSuccess ? COLA_OK : COLA_ERR_LAUNCH; }

// ------------------------------------------------------------ launch tracing
struct TraceState {
    cola_trace_slot_t* slots = nullptr;
    int32_t capacity = 0;
    int32_t* count = nullptr;
};
TraceState g_trace;

// Launch through `fn`, bracketed by the next free trace slot's events.
template <class Fn>
cudaError_t traced(int kind, int64_t m, int64_t n, int64_t k, int splits, int flags, cudaStream_t st, Fn&& fn)
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
        slot->m = static_cast<int32_t>(m);
        slot->n = static_cast<int32_t>(n);
        slot->k = static_cast<int32_t>(k);
        slot->splits = splits;
        slot->flags = flags;
        ++*g_trace.count;
    }
    return cudaSuccess;
}

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

// ------------------------------------------------------------ passes
// F1: Z = X A^T, H = sigma(Z)  (Z pitch / H pitch ldz; N = the r columns of A given)
cola_status_t run_f1(const Shape& s, int sigma, int64_t N, const void* X, const void* A, void* Z, void* H,
                     int64_t ldz, unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn(N);
    const int ms = choose_msub(s.n, N, s.d_in, bn);
    GemmParams p = plan(s.n, N, s.d_in, bn, ms, sms, false);
    CUtensorMap ma, mb, md, md2;
    COLA_MAP(map_kmajor(&ma, X, s.d_in, s.n, s.ld_x, BM * ms));
    COLA_MAP(map_kmajor(&mb, A, s.d_in, N, s.ld_a, bn));
    COLA_MAP(map_box32(&md, Z, N, s.n, ldz));
    if (H) COLA_MAP(map_box32(&md2, H, N, s.n, ldz));
    p.has_d2 = H != nullptr;
    p.sigma = sigma;
    p.status = status;
    return launched(traced(COLA_KERNEL_FWD_ZH, s.n, N, s.d_in, 1, H != nullptr, st, [&] {
        return dispatch<false, false, EPI_ZH>(bn, ms, ma, mb, md, H ? md2 : md, md, p, sms, st);
    }));
}

// F2: Y = H B^T  (H [n x r] with pitch ldh)
cola_status_t run_f2(const Shape& s, const void* H, int64_t ldh, const void* B, void* Y, unsigned int* status,
                     int sms, cudaStream_t st)
{
    const int bn = choose_bn(s.d_out);
    const int ms = choose_msub(s.n, s.d_out, s.r, bn);
    GemmParams p = plan(s.n, s.d_out, s.r, bn, ms, sms, false);
    CUtensorMap ma, mb, md;
    COLA_MAP(map_kmajor(&ma, H, s.r, s.n, ldh, BM * ms));
    COLA_MAP(map_kmajor(&mb, B, s.r, s.d_out, s.r, bn));
    COLA_MAP(map_box32(&md, Y, s.d_out, s.n, s.ld_y));
    p.d_ptr = static_cast<__nv_bfloat16*>(Y);
    p.d_ld = s.ld_y;
    p.status = status;
    return launched(traced(COLA_KERNEL_FWD_Y, s.n, s.d_out, s.r, 1, 0, st, [&] {
        return dispatch<false, false, EPI_STORE>(bn, ms, ma, mb, md, md, md, p, sms, st);
    }));
}

// B1: dZ = (dY B) * sigma'(Z), and H = sigma(Z) when Hout != null (CoLA-M)
cola_status_t run_b1(const Shape& s, int sigma, const void* dY, const void* B, const void* Z, int64_t ldz,
                     void* dZ, void* Hout, unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn(s.r);
    const int ms = choose_msub(s.n, s.r, s.d_out, bn);
    GemmParams p = plan(s.n, s.r, s.d_out, bn, ms, sms, false);
    CUtensorMap ma, mb, md, md2, mz;
    COLA_MAP(map_kmajor(&ma, dY, s.d_out, s.n, s.ld_y, BM * ms));
    COLA_MAP(map_mnmajor(&mb, B, s.r, s.d_out, s.r));
    COLA_MAP(map_box32(&md, dZ, s.r, s.n, ldz));
    COLA_MAP(map_box32(&mz, Z, s.r, s.n, ldz));
    if (Hout) COLA_MAP(map_box32(&md2, Hout, s.r, s.n, ldz));
    p.has_d2 = Hout != nullptr;
    p.sigma = sigma;
    p.status = status;
    return launched(traced(COLA_KERNEL_BWD_DZ, s.n, s.r, s.d_out, 1, Hout != nullptr, st, [&] {
        return dispatch<false, true, EPI_DSIGMA>(bn, ms, ma, mb, md, Hout ? md2 : md, mz, p, sms, st);
    }));
}

// Weight gradient D[M x N] = sum_t P[t, m] Q[t, n] over the n tokens, both
// operands token-major (MN-major): split over tokens, fixed-order reduce.
cola_status_t run_wgrad(int kind, int64_t ntok, int64_t M, int64_t N, const void* P, int64_t ldp, const void* Q,
                        int64_t ldq, void* out, int64_t ldo, int accumulate_f32, float* part, size_t part_bytes,
                        unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn(N);
    const int ms = choose_msub(M, N, ntok, bn);
    GemmParams p = plan(M, N, ntok, bn, ms, sms, true);
    const int64_t slab = partial_elems(p, bn, ms);
    if (static_cast<size_t>(p.splits) * slab * 4 > part_bytes) return COLA_ERR_WORKSPACE;
    CUtensorMap ma, mb;
    COLA_MAP(map_mnmajor(&ma, P, M, ntok, ldp));
    COLA_MAP(map_mnmajor(&mb, Q, N, ntok, ldq));
    p.status = status;
    if (p.splits == 1 && !accumulate_f32) {
        // no token split: the epilogue writes the bf16 gradient directly
        CUtensorMap md;
        COLA_MAP(map_box32(&md, out, N, M, ldo));
        p.d_ptr = static_cast<__nv_bfloat16*>(out);
        p.d_ld = ldo;
        return launched(traced(kind, M, N, ntok, 1, 0, st,
                               [&] { return dispatch<true, true, EPI_STORE>(bn, ms, ma, mb, md, md, md, p, sms, st); }));
    }
    p.D = part;
    p.ldd = p.n_tiles * bn;
    p.part_stride = slab;
    COLA_TRY(launched(traced(kind, M, N, ntok, p.splits, 0, st,
                             [&] { return dispatch<true, true, EPI_F32>(bn, ms, ma, mb, ma, ma, ma, p, sms, st); })));
    return launched(traced(COLA_KERNEL_REDUCE, M, N, p.splits, p.splits, 0, st, [&] {
        return launch_splitk_reduce(part, p.splits, slab, p.n_tiles * bn, static_cast<int>(M), static_cast<int>(N),
                                    out, ldo, accumulate_f32, sms * 4, st);
    }));
}

// B4: dX = dZ A  (dZ [n x K] pitch ldz, A [K x d_in] pitch ld_a; K = r or 3r)
cola_status_t run_b4(const Shape& s, int64_t K, const void* dZ, int64_t ldz, const void* A, void* dX,
                     unsigned int* status, int sms, cudaStream_t st)
{
    const int bn = choose_bn(s.d_in);
    const int ms = choose_msub(s.n, s.d_in, K, bn);
    GemmParams p = plan(s.n, s.d_in, K, bn, ms, sms, false);
    CUtensorMap ma, mb, md;
    COLA_MAP(map_kmajor(&ma, dZ, K, s.n, ldz, BM * ms));
    COLA_MAP(map_mnmajor(&mb, A, s.d_in, K, s.ld_a));
    COLA_MAP(map_box32(&md, dX, s.d_in, s.n, s.ld_x));
    p.d_ptr = static_cast<__nv_bfloat16*>(dX);
    p.d_ld = s.ld_x;
    p.status = status;
    return launched(traced(COLA_KERNEL_BWD_DX, s.n, s.d_in, K, 1, 0, st, [&] {
        return dispatch<false, true, EPI_STORE>(bn, ms, ma, mb, md, md, md, p, sms, st);
    }));
}

}  // namespace
}  // namespace cola

using namespace cola;

extern "C" {

cola_status_t cola_workspace_size(const cola_desc_t* desc, int fused_qkv, size_t* bytes)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    if (!bytes || (fused_qkv != 0 && fused_qkv != 1)) return COLA_ERR_INVALID;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    *bytes = ws_layout(*desc, fused_qkv, sms).total;
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
    COLA_TRY(check_ptrs({X, A, B, Y, Z_save}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_save != nullptr : H_save == nullptr) return COLA_ERR_INVALID;
    if (H_save && !aligned16(H_save)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 0, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    void* H = cola_m ? static_cast<void*>(wsb(ws) + L.h_off) : H_save;
    COLA_TRY(run_f1(s, desc->sigma, s.r, X, A, Z_save, H, s.r, status, sms, st));
    return run_f2(s, H, s.r, B, Y, status, sms, st);
}

cola_status_t cola_bwd(const cola_desc_t* desc, const void* X, const void* A, const void* B, const void* dY,
                       const void* Z_save, const void* H_save, void* dX, void* dA, void* dB, void* ws,
                       size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    COLA_TRY(check_ptrs({X, A, B, dY, Z_save, dX, dA, dB}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_save != nullptr : H_save == nullptr) return COLA_ERR_INVALID;
    if (H_save && !aligned16(H_save)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 0, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    void* dZ = wsb(ws) + L.dz_off;
    void* Hrec = cola_m ? static_cast<void*>(wsb(ws) + L.h_off) : nullptr;
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    const int acc = desc->wgrad_fp32;

    COLA_TRY(run_b1(s, desc->sigma, dY, B, Z_save, s.r, dZ, Hrec, status, sms, st));
    const void* Hsrc = cola_m ? Hrec : H_save;
    COLA_TRY(run_wgrad(COLA_KERNEL_WGRAD_DB, s.n, s.d_out, s.r, dY, s.ld_y, Hsrc, s.r, dB, s.r, acc, part, part_bytes, status, sms, st));
    COLA_TRY(run_wgrad(COLA_KERNEL_WGRAD_DA, s.n, s.r, s.d_in, dZ, s.r, X, s.ld_x, dA, s.ld_a, acc, part, part_bytes, status, sms, st));
    return run_b4(s, s.r, dZ, s.r, A, dX, status, sms, st);
}

cola_status_t cola_fwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, void* Y_q, void* Y_k, void* Y_v, void* Z_qkv,
                                 void* H_qkv, void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    COLA_TRY(check_ptrs({X, A_qkv, B_q, B_k, B_v, Y_q, Y_k, Y_v, Z_qkv}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_qkv != nullptr : H_qkv == nullptr) return COLA_ERR_INVALID;
    if (H_qkv && !aligned16(H_qkv)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 1, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = 3 * s.r;
    uint8_t* H = cola_m ? wsb(ws) + L.h_off : static_cast<uint8_t*>(H_qkv);
    COLA_TRY(run_f1(s, desc->sigma, R, X, A_qkv, Z_qkv, H, R, status, sms, st));
    const void* Bs[3] = {B_q, B_k, B_v};
    void* Ys[3] = {Y_q, Y_k, Y_v};
    for (int j = 0; j < 3; ++j)
        COLA_TRY(run_f2(s, H + static_cast<size_t>(j) * s.r * 2, R, Bs[j], Ys[j], status, sms, st));
    return COLA_OK;
}

cola_status_t cola_bwd_qkv_fused(const cola_desc_t* desc, const void* X, const void* A_qkv, const void* B_q,
                                 const void* B_k, const void* B_v, const void* dY_q, const void* dY_k,
                                 const void* dY_v, const void* Z_qkv, const void* H_qkv, void* dX, void* dA_qkv,
                                 void* dB_q, void* dB_k, void* dB_v, void* ws, size_t ws_bytes, void* stream)
{
    Shape s;
    COLA_TRY(check_desc(desc, &s));
    COLA_TRY(check_ptrs({X, A_qkv, B_q, B_k, B_v, dY_q, dY_k, dY_v, Z_qkv, dX, dA_qkv, dB_q, dB_k, dB_v}));
    const bool cola_m = desc->mode == COLA_MODE_COLA_M;
    if (cola_m ? H_qkv != nullptr : H_qkv == nullptr) return COLA_ERR_INVALID;
    if (H_qkv && !aligned16(H_qkv)) return COLA_ERR_ALIGN;
    int sms = 0;
    COLA_TRY(device_info(&sms));
    WsLayout L;
    COLA_TRY(check_ws(*desc, 1, sms, ws, ws_bytes, &L));
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    unsigned int* status = ws_status(ws);
    const int64_t R = 3 * s.r;
    const size_t slice = static_cast<size_t>(s.r) * 2;   // bytes between the q, k, v column blocks
    uint8_t* dZ = wsb(ws) + L.dz_off;
    uint8_t* Hrec = cola_m ? wsb(ws) + L.h_off : nullptr;
    float* part = reinterpret_cast<float*>(wsb(ws) + L.part_off);
    const size_t part_bytes = L.total - L.part_off;
    const int acc = desc->wgrad_fp32;
    const void* Bs[3] = {B_q, B_k, B_v};
    const void* dYs[3] = {dY_q, dY_k, dY_v};
    void* dBs[3] = {dB_q, dB_k, dB_v};
    const uint8_t* Zb = static_cast<const uint8_t*>(Z_qkv);
    const uint8_t* Hsrc = cola_m ? Hrec : static_cast<const uint8_t*>(H_qkv);
    for (int j = 0; j < 3; ++j) {
        COLA_TRY(run_b1(s, desc->sigma, dYs[j], Bs[j], Zb + j * slice, R, dZ + j * slice,
                        Hrec ? Hrec + j * slice : nullptr, status, sms, st));
        COLA_TRY(run_wgrad(COLA_KERNEL_WGRAD_DB, s.n, s.d_out, s.r, dYs[j], s.ld_y, Hsrc + j * slice, R, dBs[j], s.r, acc, part,
                           part_bytes, status, sms, st));
    }
    COLA_TRY(run_wgrad(COLA_KERNEL_WGRAD_DA, s.n, R, s.d_in, dZ, R, X, s.ld_x, dA_qkv, s.ld_a, acc, part, part_bytes, status, sms, st));
    return run_b4(s, R, dZ, R, A_qkv, dX, status, sms, st);
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
