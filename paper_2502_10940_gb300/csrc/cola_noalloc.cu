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
// device current, on the first call that runs on it; kernels only ever see
// that address.
#include <cuda_runtime.h>

#include <cstdint>
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

struct ScratchSlot {
    std::once_flag once;
    cudaError_t err = cudaSuccess;
    void* ptr = nullptr;
};
ScratchSlot g_slots[64];

// Device address of g_wgrad_scratch on the current device (set up once per device).
cudaError_t scratch_address(int dev, void** out)
{
    ScratchSlot& s = g_slots[dev];
    std::call_once(s.once, [&] {
        void* p = nullptr;
        s.err = cudaGetSymbolAddress(&p, g_wgrad_scratch);
        if (s.err == cudaSuccess) s.ptr = p;
    });
    *out = s.ptr;
    return s.err;
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
    const int bn = choose_bn(N);
    const int ms = choose_msub(M, N, n_tokens, bn);
    GemmParams p = plan(M, N, n_tokens, bn, ms, sms, true);
    const int64_t slab = partial_elems(p, bn, ms);
    const size_t slab_bytes = static_cast<size_t>(slab) * 4;
    if (slab_bytes > kStaticScratchBytes) return COLA_ERR_WORKSPACE;   // too large even unsplit
    const int max_splits = static_cast<int>(kStaticScratchBytes / slab_bytes);
    if (p.splits > max_splits) {
        p.kb_per_split = (p.k_blocks + max_splits - 1) / max_splits;
        p.splits = (p.k_blocks + p.kb_per_split - 1) / p.kb_per_split;
        p.units = p.m_tiles * p.n_tiles * p.splits;
    }

    // ---- set-up: the scratch's device address on this device (first call only)
    void* scratch = nullptr;
    if (scratch_address(dev, &scratch) != cudaSuccess || scratch == nullptr) return COLA_ERR_LAUNCH;

    CUtensorMap ma, mb;
    if (!map_mnmajor(&ma, P, M, n_tokens, ld_p) || !map_mnmajor(&mb, Q, N, n_tokens, ld_q)) return COLA_ERR_LAUNCH;
    float* part = static_cast<float*>(scratch);
    p.D = part;
    p.ldd = p.n_tiles * bn;
    p.part_stride = slab;
    p.status = nullptr;   // no workspace to report a device-side timeout through
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (dispatch<true, true, EPI_F32>(bn, ms, ma, mb, ma, ma, ma, p, sms, st) != cudaSuccess) return COLA_ERR_LAUNCH;
    if (launch_splitk_reduce(part, p.splits, slab, p.n_tiles * bn, static_cast<int>(M), static_cast<int>(N), D, ld_d,
                             accumulate_f32, sms * 4, st) != cudaSuccess)
        return COLA_ERR_LAUNCH;
    return COLA_OK;
}
