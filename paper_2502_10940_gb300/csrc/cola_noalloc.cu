// cola_noalloc.cu -- cola_wgrad_static_scratch: the weight-gradient GEMM of a
// CoLA factor for callers that cannot allocate device memory.
//
// Some callers can pass the library only the tensors they operate on: a
// plugin or operator interface whose signature carries inputs and outputs
// but no workspace, or a process whose device memory is fixed at start-up by
// another allocator, so that any later cudaMalloc would fail or break the
// caller's budget.  cola_bwd needs a caller-owned workspace for the token
// split of its weight gradients; this entry point keeps that scratch in a
// file-scope device array instead, sized once at library load.
//
// The array's name is only a host-side stand-in in host code.  Its device
// address is fetched with cudaGetSymbolAddress once per device, with that
// device current, on the first call that runs on it (a failed lookup is
// retried by the next call); kernels only ever see that address.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "cola.h"
#include "gemm_launch.cuh"
#include "host_plan.cuh"

namespace cola {
namespace {

constexpr size_t kStaticScratchBytes = static_cast<size_t>(COLA_STATIC_SCRATCH_BYTES);

// fp32 token-split partial slabs of one weight gradient; shared by every call
// on a device (calls that overlap on the GPU race on it).
static __device__ __align__(256) unsigned char g_wgrad_scratch[kStaticScratchBytes];

// Per device, the array's device address once a lookup has succeeded; a
// failed lookup is not cached, so the next call on that device tries again.
std::atomic<void*> g_scratch_ptr[64];
std::mutex g_scratch_mu;

// Device address of g_wgrad_scratch on the current device `dev`.
cudaError_t scratch_address(int dev, void** out)
{
    void* p = g_scratch_ptr[dev].load(std::memory_order_acquire);
    if (!p) {
        std::lock_guard<std::mutex> lock(g_scratch_mu);
        p = g_scratch_ptr[dev].load(std::memory_order_relaxed);
        if (!p) {
            const cudaError_t e = cudaGetSymbolAddress(&p, g_wgrad_scratch);
            if (e != cudaSuccess) return e;
            if (!p) return cudaErrorInvalidSymbol;
            g_scratch_ptr[dev].store(p, std::memory_order_release);
        }
    }
    *out = p;
    return cudaSuccess;
}

}  // namespace
}  // namespace cola

using namespace cola;

extern "C" cola_status_t cola_wgrad_static_scratch(int64_t n_tokens, int64_t M, int64_t N, const void* P,
                                                   int64_t ld_p, const void* Q, int64_t ld_q, void* D, int64_t ld_d,
                                                   int32_t accumulate_f32, void* stream)
{
    // ---- argument checks (nothing touches the device before they pass)
    if (!P || !Q || !D) return COLA_ERR_INVALID;
    if (n_tokens < 1 || M < 1 || N < 1) return COLA_ERR_INVALID;
    if (accumulate_f32 != 0 && accumulate_f32 != 1) return COLA_ERR_INVALID;
    if (ld_p < M || ld_q < N || ld_d < N || ld_p % 8 || ld_q % 8 || (!accumulate_f32 && ld_d % 8) ||
        (accumulate_f32 && ld_d % 4))
        return COLA_ERR_INVALID;
    if (((reinterpret_cast<uintptr_t>(P) | reinterpret_cast<uintptr_t>(Q) | reinterpret_cast<uintptr_t>(D)) & 15u) != 0)
        return COLA_ERR_ALIGN;
    const int64_t lim = (int64_t(1) << 31) - 256;
    if (n_tokens > lim || M > lim || N > lim || ld_p > lim || ld_q > lim || ld_d > lim) return COLA_ERR_UNSUPPORTED;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return COLA_ERR_LAUNCH;
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return COLA_ERR_LAUNCH;
    if (major != 10 || minor != 3) return COLA_ERR_UNSUPPORTED;

    // ---- plan; shrink the token split until its partials fit the static scratch
    const int64_t Ms[1] = {M}, Ns[1] = {N};
    WgradPlan w = plan_wgrad(Ms, Ns, 1, n_tokens, sms);
    const size_t slab_bytes = static_cast<size_t>(w.slab[0]) * 4;
    if (slab_bytes > kStaticScratchBytes) return COLA_ERR_WORKSPACE;   // too large even unsplit
    const int max_splits = static_cast<int>(kStaticScratchBytes / slab_bytes);
    if (w.p[0].splits > max_splits) set_splits(w.p[0], max_splits);

    cudaStream_t st = static_cast<cudaStream_t>(stream);
    GemmBatch b;
    std::memset(&b, 0, sizeof b);
    b.count = 1;
    GemmProblem& pr = b.prob[0];
    pr.p = w.p[0];
    if (!map_mnmajor(&pr.map_a, P, M, n_tokens, ld_p) || !map_mnmajor(&pr.map_b, Q, N, n_tokens, ld_q))
        return COLA_ERR_LAUNCH;
    pr.p.status = nullptr;   // no workspace to report a device-side timeout through
    if (pr.p.splits == 1 && !accumulate_f32) {
        // unsplit: the epilogue stores the bf16 gradient directly; no scratch
        if (!map_box32(&pr.map_d, D, N, M, ld_d)) return COLA_ERR_LAUNCH;
        pr.map_d2 = pr.map_z = pr.map_d;
        pr.p.d_ptr = static_cast<__nv_bfloat16*>(D);
        pr.p.d_ld = ld_d;
        return dispatch<true, true, EPI_STORE>(w.bn, w.msub, b, sms, st) == cudaSuccess ? COLA_OK : COLA_ERR_LAUNCH;
    }

    // ---- set-up: the scratch's device address on this device (first call only)
    void* scratch = nullptr;
    if (scratch_address(dev, &scratch) != cudaSuccess || scratch == nullptr) return COLA_ERR_LAUNCH;

    pr.map_d = pr.map_d2 = pr.map_z = pr.map_a;
    float* part = static_cast<float*>(scratch);
    pr.p.D = part;
    pr.p.ldd = static_cast<long long>(pr.p.n_tiles) * w.bn;
    pr.p.part_stride = w.slab[0];
    if (dispatch<true, true, EPI_F32>(w.bn, w.msub, b, sms, st) != cudaSuccess) return COLA_ERR_LAUNCH;
    ReduceBatch rb;
    std::memset(&rb, 0, sizeof rb);
    rb.count = 1;
    rb.splits = pr.p.splits;
    rb.accumulate_f32 = accumulate_f32;
    rb.job[0].part = part;
    rb.job[0].part_stride = w.slab[0];
    rb.job[0].ldp = pr.p.n_tiles * w.bn;
    rb.job[0].M = static_cast<int>(M);
    rb.job[0].N = static_cast<int>(N);
    rb.job[0].out = D;
    rb.job[0].ldo = ld_d;
    if (launch_splitk_reduce(rb, st) != cudaSuccess) return COLA_ERR_LAUNCH;
    return COLA_OK;
}
