// logq_quantize_noalloc: logq_quantize for callers that cannot allocate device
// memory.  Some programs must not call cudaMalloc from this library: a plugin
// running inside a host application that owns every device allocation through
// its own pool (and budgets it), or a latency-critical path that cannot take
// the implicit device synchronisation of an allocation.  Such a caller cannot
// hand logq_quantize the workspace it needs, so this entry point keeps that
// scratch record in a static device array of the library instead; the
// quantisation itself is logq_quantize's (logq::quantize_with).
//
// The array below is the scratch: one 256-byte record (the absmax word and the
// non-finite flag of the quantiser).  Every GPU that loads the library holds
// one copy until the process exits.  Host code may not use the array's name as
// an address (on the host it names a stand-in, not device memory); its device
// address is looked up with cudaGetSymbolAddress, with the device current, once
// per device and CUDA context (a context created after a reset of the device
// gets a fresh lookup).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <string.h>

#include <mutex>

#include "internal.h"

namespace {

constexpr size_t kStaticScratchBytes = 256;   // maximum scratch of this entry point

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

// Driver calls that name the current context (through the runtime's
// entry-point lookup, so the library needs no link against libcuda).
struct CtxFns {
    PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
    PFN_cuCtxGetId_v12000 get_id = nullptr;
};

const CtxFns& ctx_fns()
{
    static CtxFns f;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            f.get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            f.get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
    });
    return f;
}

// Device address of g_static_scratch in the current device's context, looked
// up the first time a device (or a new context on it) is seen, and cached by
// device and context id.
cudaError_t static_scratch(logq::Workspace** out)
{
    static std::mutex mu;
    static void* addr[64] = {nullptr};
    static unsigned long long ctx_id[64] = {0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    const CtxFns& f = ctx_fns();
    if (!f.get_current || !f.get_id) return cudaErrorInitializationError;
    auto current_id = [&](unsigned long long* id) -> bool {
        CUcontext ctx = nullptr;
        return f.get_current(&ctx) == CUDA_SUCCESS && ctx && f.get_id(ctx, id) == CUDA_SUCCESS;
    };
    std::lock_guard<std::mutex> g(mu);
    unsigned long long id = 0;
    const bool have_ctx = current_id(&id);
    if (!have_ctx || addr[dev] == nullptr || ctx_id[dev] != id) {
        // set-up for this device and context (the lookup also makes the
        // device's primary context current when none is yet)
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        if (!current_id(&id)) return cudaErrorInitializationError;
        addr[dev] = p;
        ctx_id[dev] = id;
    }
    *out = static_cast<logq::Workspace*>(addr[dev]);
    return cudaSuccess;
}

}  // namespace

extern "C" logq_status logq_quantize_noalloc(const float* W, int64_t N, int64_t K, int bits,
                                             double base, double range, int flags, uint8_t* codes,
                                             logq_codebook* cb_out, void* stream)
{
    using namespace logq;
    const logq_status st = check_quantize_args(W, N, K, bits, base, range, flags, codes);
    if (st != LOGQ_OK) return st;
    // The scratch needed does not grow with N or K; it is one workspace record.
    if (kWorkspaceBytes > kStaticScratchBytes) return LOGQ_ERR_WORKSPACE;
    Workspace* ws = nullptr;
    if (static_scratch(&ws) != cudaSuccess) return LOGQ_ERR_CUDA;
    // The array keeps the previous call's words: quantize_with clears the two it uses.
    return quantize_with(W, N, K, bits, base, range, flags, codes, cb_out, ws, static_cast<cudaStream_t>(stream));
}
