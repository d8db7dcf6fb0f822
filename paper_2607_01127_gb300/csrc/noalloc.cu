// logq_quantize_noalloc: logq_quantize for callers that cannot allocate device
// memory.  Some programs must not call cudaMalloc from this library: a plugin
// running inside a host application that owns every device allocation through
// its own pool (and budgets it), or a latency-critical path that cannot take
// the implicit device synchronisation of an allocation.  Such a caller cannot
// hand logq_quantize the workspace it needs, so this entry point keeps that
// scratch record in a static device array of the library instead.
//
// The array below is the scratch: one 256-byte record (the absmax word and the
// non-finite flag of the quantiser).  Every GPU that loads the library holds
// one copy until the process exits.  Host code may not use the array's name as
// an address (on the host it names a stand-in, not device memory); its device
// address is looked up once per device with cudaGetSymbolAddress.
#include <cuda_runtime.h>
#include <math.h>
#include <string.h>

#include <mutex>

#include "internal.h"

namespace {

constexpr size_t kStaticScratchBytes = 256;   // maximum scratch of this entry point

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Device address of g_static_scratch on the current device, looked up on the
// first call per device (with that device current) and cached.
cudaError_t static_scratch(logq::Workspace** out)
{
    static std::mutex mu;
    static void* addr[64] = {nullptr};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> g(mu);
    if (addr[dev] == nullptr) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
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
    if (!W || !codes || !aligned16(W) || !aligned16(codes)) return LOGQ_ERR_INVALID_ARG;
    if (logq_packed_bytes(N, K, bits) == 0) return LOGQ_ERR_INVALID_ARG;
    if (!isfinite(base) || !(base > 1.0) || isnan(range) || isinf(range)) return LOGQ_ERR_INVALID_ARG;
    if (flags != LOGQ_SHIFT_EXACT && flags != LOGQ_SHIFT_FLOOR) return LOGQ_ERR_INVALID_ARG;
    if (N > (int64_t(1) << 40) / K) return LOGQ_ERR_INVALID_ARG;
    // The scratch needed does not grow with N or K; it is one workspace record.
    if (kWorkspaceBytes > kStaticScratchBytes) return LOGQ_ERR_WORKSPACE;

    Workspace* ws = nullptr;
    if (static_scratch(&ws) != cudaSuccess) return LOGQ_ERR_CUDA;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // The array keeps the previous call's words: clear the two this call uses.
    if (cudaMemsetAsync(ws, 0, 2 * sizeof(uint32_t), s) != cudaSuccess) return LOGQ_ERR_CUDA;

    uint32_t host_words[2] = {0, 0};
    const bool auto_range = !(range > 0.0);
    if (auto_range) {
        if (launch_absmax(W, N * K, ws, s) != cudaSuccess) return LOGQ_ERR_CUDA;
        if (cudaMemcpyAsync(host_words, ws, sizeof host_words, cudaMemcpyDeviceToHost, s) != cudaSuccess)
            return LOGQ_ERR_CUDA;
        if (cudaStreamSynchronize(s) != cudaSuccess) return LOGQ_ERR_CUDA;
        if (host_words[1]) return LOGQ_ERR_NONFINITE;
        float mx;
        memcpy(&mx, &host_words[0], 4);
        if (!(mx > 0.0f)) return LOGQ_ERR_INVALID_ARG;
        range = (double)mx;
    }
    logq_codebook cb;
    const logq_status st = logq_build_codebook(bits, base, range, flags, &cb);
    if (st != LOGQ_OK) return st;
    QuantParams p;
    memset(&p, 0, sizeof p);
    for (int j = 0; j < 128; ++j) p.thresh[j] = cb.thresh[j];
    p.qmax = cb.qmax;
    p.bits = bits;
    p.check_nonfinite = auto_range ? 0 : 1;
    if (launch_quantize(W, N, K, p, codes, ws, s) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (cudaMemcpyAsync(host_words, ws, sizeof host_words, cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return LOGQ_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (!auto_range && host_words[1]) return LOGQ_ERR_NONFINITE;
    if (cb_out) *cb_out = cb;
    return LOGQ_OK;
}
