// Internal declarations shared by the translation units of liblogq.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "logq.h"

namespace logq {

// Workspace layout (logq_workspace_bytes() bytes, caller-allocated, zeroed once).
struct Workspace {
    uint32_t absmax_bits;   // max |w| as fp32 bits (atomicMax over non-negative floats)
    uint32_t nonfinite;     // 1 when a NaN / Inf weight was seen
    uint32_t error;         // device error word: LOGQ_ERR_TIMEOUT when a wait gave up
    uint32_t detail;        // which wait gave up (implementation code)
    uint32_t reserved[60];
};
static_assert(sizeof(Workspace) == 256, "workspace layout");
constexpr size_t kWorkspaceBytes = sizeof(Workspace);

// Device state of the energy-range selection (caller-provided scratch,
// logq_energy_scratch_bytes() bytes): bucket energies of the current level as
// exact integer sums of the high / low 24 bits of m^2, the total energy, the
// energy below the selected prefix, the prefix and the result.
struct EnergyState {
    unsigned long long hi[4096];
    unsigned long long lo[4096];
    double total;
    double below;
    uint32_t prefix;
    uint32_t wmin_bits;
    uint32_t failed;        // the window pass found the crossing below its window
    uint32_t _pad;
};

// Decision boundaries handed to the quantise kernel (fp32, rounded up).
struct QuantParams {
    float thresh[128];
    int32_t qmax;
    int32_t bits;
    int32_t check_nonfinite;
    int32_t _pad;
};

// One quantised linear call after validation.
struct LinearArgs {
    const uint8_t* codes;
    const void* X;
    void* Y;
    int64_t B, N, K;
    int bits;
    int x_f16;              // 0: bf16 activations, 1: fp16
    int y_dtype;            // logq_dtype of Y
    uint16_t lvl16[256];    // code-indexed 16-bit levels in X's dtype (2^bits used)
    Workspace* ws;
    size_t ws_bytes;        // the caller's workspace bytes (beyond kWorkspaceBytes: split-k partial sums)
};

// A grouped launch (decode GEMV or tensor-core prefill): up to four matrices
// that share X (e.g. q/k/v or gate/up), each with its own codebook and output.
struct GroupItem {
    const uint8_t* codes;
    void* Y;
    int64_t N;
    uint16_t lvl16[256];
};

struct GroupArgs {
    GroupItem item[4];
    int count;
    const void* X;
    int64_t B, K;
    int bits;
    int x_f16;
    int y_dtype;
    const void* pf;          // optional L2 warm-up range
    int64_t pf_bytes;
    Workspace* ws;
};

// The part of a prefetch hint [p, p + bytes) that a bulk L2 prefetch may take:
// the start rounded up to 16 bytes and the length down to a multiple of 16 that
// stays inside the range (*start = nullptr, *len = 0 when nothing is left).
inline void aligned_prefetch_range(const void* p, size_t bytes, const void** start, int64_t* len)
{
    const uintptr_t p0 = reinterpret_cast<uintptr_t>(p);
    const uintptr_t a = (p0 + 15u) & ~(uintptr_t)15u;
    const size_t skip = (size_t)(a - p0);
    const size_t n = (p && bytes > skip) ? ((bytes - skip) / 16) * 16 : 0;
    *start = n > 0 ? reinterpret_cast<const void*>(a) : nullptr;
    *len = (int64_t)n;
}

int sm_count();
// logq_quantize after its workspace check: argument checks, and the
// quantisation on a given workspace record (shared with the allocation-free
// entry point, which passes its static record).
logq_status check_quantize_args(const float* W, int64_t N, int64_t K, int bits, double base, double range,
                                int flags, const uint8_t* codes);
logq_status quantize_with(const float* W, int64_t N, int64_t K, int bits, double base, double range, int flags,
                          uint8_t* codes, logq_codebook* cb_out, Workspace* ws, cudaStream_t s);
cudaError_t launch_absmax(const float* W, int64_t count, Workspace* ws, cudaStream_t s);
cudaError_t launch_energy_range(const float* W, int64_t count, double eps, EnergyState* st, Workspace* ws,
                                cudaStream_t s);
cudaError_t launch_quantize(const float* W, int64_t N, int64_t K, const QuantParams& p,
                            uint8_t* codes, Workspace* ws, cudaStream_t s);
cudaError_t launch_gemv(const LinearArgs& a, cudaStream_t s);
size_t gptq_scratch_bytes(int64_t N, int64_t K);
cudaError_t launch_gptq(const float* W, int64_t N, int64_t K, const float* U, const uint8_t* dead, int bits,
                        const float* thresh, const float* level, int qmax, uint8_t* codes, void* scratch,
                        cudaStream_t s);
size_t gptq_factor_scratch_bytes(int64_t K);
cudaError_t launch_gptq_factor(const float* H, int64_t K, double damp, float* U, uint8_t* dead, void* scratch,
                               uint32_t* not_pd, cudaStream_t s);
cudaError_t launch_gemv_group(const GroupArgs& a, cudaStream_t s);
cudaError_t launch_prefill(const LinearArgs& a, cudaStream_t s);
// One tensor-core launch over the group's matrices (ws_bytes: the caller's
// workspace, which holds the split k ranges' partial sums).
cudaError_t launch_prefill_group(const GroupArgs& g, size_t ws_bytes, cudaStream_t s);
// Tensor-core launch plan of B x N[i] x K products sharing X (count <= 4):
// token-tile width, k ranges per output tile (the partial sums need part_bytes
// of workspace beyond kWorkspaceBytes; at most part_bytes_avail are used) and
// the CTAs each matrix gets.
struct PrefillPlan {
    int bn;
    int splits;
    int ksplit;
    size_t part_bytes;
    double est_us;          // estimated launch time on a GB300 (planning only)
    int ncta[4];
};
PrefillPlan prefill_plan(int64_t B, const int64_t* N, int count, int64_t K, size_t part_bytes_avail);
PrefillPlan prefill_plan(int64_t B, int64_t N, int64_t K, size_t part_bytes_avail);
bool gemv_supports(int bits, int64_t B);

}  // namespace logq
