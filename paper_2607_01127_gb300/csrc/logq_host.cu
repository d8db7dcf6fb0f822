// C-ABI front of liblogq: argument validation, the host codebook builder
// (paper Sec. 3.1, Eqs. (2) and (4)) and dispatch to the device kernels.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math.h>
#include <string.h>

#include <mutex>

#include "internal.h"

namespace logq {

int sm_count()
{
    static int cached[64] = {0};
    static std::mutex mu;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> g(mu);
    if (cached[dev] == 0) {
        int v = 0;
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        cached[dev] = v;
    }
    return cached[dev];
}

// Argument checks shared by logq_quantize and logq_quantize_noalloc (all but
// the scratch, which the two take from different places).
logq_status check_quantize_args(const float* W, int64_t N, int64_t K, int bits, double base, double range,
                                int flags, const uint8_t* codes)
{
    if (!W || !codes || (reinterpret_cast<uintptr_t>(W) & 15u) || (reinterpret_cast<uintptr_t>(codes) & 15u))
        return LOGQ_ERR_INVALID_ARG;
    if (logq_packed_bytes(N, K, bits) == 0) return LOGQ_ERR_INVALID_ARG;
    if (!isfinite(base) || !(base > 1.0) || isnan(range) || isinf(range)) return LOGQ_ERR_INVALID_ARG;
    if (flags != LOGQ_SHIFT_EXACT && flags != LOGQ_SHIFT_FLOOR) return LOGQ_ERR_INVALID_ARG;
    if (N > (int64_t(1) << 40) / K) return LOGQ_ERR_INVALID_ARG;
    return LOGQ_OK;
}

// The quantisation itself, on a workspace record ws (device): Sec. 3.2 w_max
// when range <= 0, the codebook (Eqs. (2), (4)), then Eq. (1) and packing;
// one 8-byte readback and one stream synchronisation report non-finite
// weights.  Clears the two workspace words it uses first.
logq_status quantize_with(const float* W, int64_t N, int64_t K, int bits, double base, double range, int flags,
                          uint8_t* codes, logq_codebook* cb_out, Workspace* ws, cudaStream_t s)
{
    cudaError_t e = cudaMemsetAsync(ws, 0, 2 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return LOGQ_ERR_CUDA;

    uint32_t host_words[2] = {0, 0};
    const bool auto_range = !(range > 0.0);
    if (auto_range) {
        // Sec. 3.2: w_max = max_i |w_i|, reduced on the device.
        if ((e = launch_absmax(W, N * K, ws, s)) != cudaSuccess) return LOGQ_ERR_CUDA;
        if ((e = cudaMemcpyAsync(host_words, ws, sizeof host_words, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
            return LOGQ_ERR_CUDA;
        if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return LOGQ_ERR_CUDA;
        if (host_words[1]) return LOGQ_ERR_NONFINITE;
        float mx;
        memcpy(&mx, &host_words[0], 4);
        if (!(mx > 0.0f)) return LOGQ_ERR_INVALID_ARG;   // all-zero weights: no log range
        range = (double)mx;
    }

    logq_codebook cb;
    logq_status st = logq_build_codebook(bits, base, range, flags, &cb);
    if (st != LOGQ_OK) return st;

    QuantParams p;
    memset(&p, 0, sizeof p);
    for (int j = 0; j < 128; ++j) p.thresh[j] = cb.thresh[j];
    p.qmax = cb.qmax;
    p.bits = bits;
    p.check_nonfinite = auto_range ? 0 : 1;
    if ((e = launch_quantize(W, N, K, p, codes, ws, s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (!auto_range) {
        if ((e = cudaMemcpyAsync(host_words, ws, sizeof host_words, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
            return LOGQ_ERR_CUDA;
        if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return LOGQ_ERR_CUDA;
        if (host_words[1]) return LOGQ_ERR_NONFINITE;
    } else {
        if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    }
    if (cb_out) *cb_out = cb;
    return LOGQ_OK;
}

}  // namespace logq

using namespace logq;

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Largest integer e with b^e <= x (x > 0, b > 1), settled with exact power
// comparisons so that exact powers of b are not lost to rounding of log().
long floor_log_base(double x, double b)
{
    long e = (long)floor(log(x) / log(b));
    while (pow(b, (double)(e + 1)) <= x) ++e;
    while (pow(b, (double)e) > x) --e;
    return e;
}

// Smallest fp32 >= t for t > 0.
float round_up_f32(double t)
{
    float f = (float)t;
    while ((double)f < t) f = nextafterf(f, INFINITY);
    for (;;) {
        float g = nextafterf(f, 0.0f);
        if ((double)g >= t) f = g;
        else break;
    }
    return f;
}

uint16_t bf16_bits_of(float v)
{
    __nv_bfloat16 h = __float2bfloat16_rn(v);
    uint16_t b;
    memcpy(&b, &h, 2);
    return b;
}

uint16_t f16_bits_of(float v)
{
    __half h = __float2half_rn(v);
    uint16_t b;
    memcpy(&b, &h, 2);
    return b;
}

logq_status cuda_status(cudaError_t e) { return e == cudaSuccess ? LOGQ_OK : LOGQ_ERR_CUDA; }

// 4-bit batches from this size up to 16 may run on the tensor cores instead of
// the CUDA-core skinny GEMM (whose fp32 FMAs bound it at 16 per weight).
#ifndef LOGQ_TC_MIN_BATCH
#define LOGQ_TC_MIN_BATCH 8
#endif

// Batches that always run on the tensor cores, or may (4-bit, LOGQ_TC_MIN_BATCH..16).
bool tensor_core_batch(int bits, int64_t B)
{
    return !gemv_supports(bits, B) || (bits == 4 && B >= LOGQ_TC_MIN_BATCH && B <= 16);
}

// A 4-bit batch of LOGQ_TC_MIN_BATCH..16 takes the tensor cores when their
// estimated time beats the CUDA-core kernel's: ~27 us per 58.7 M weights at
// batches up to 8 and ~49 us at 9..16 (the batch is padded to 8 or 16; fp32
// FMAs bound it), plus ~2 us per launch (measured on the GB300 on the
// Llama-3.1-8B shapes).  The tensor-core estimate depends on how far the caller's
// workspace lets the k ranges split (prefill_plan).
double cuda_core_us(int64_t B, int64_t N, int64_t K)
{
    return (double)N * (double)K * (B <= 8 ? 0.46e-6 : 0.84e-6) + 2.0;
}

bool use_small_batch_tc(int bits, int64_t B, int64_t N, int64_t K, size_t workspace_bytes)
{
    if (!(bits == 4 && B >= LOGQ_TC_MIN_BATCH && B <= 16)) return false;
    const size_t avail = workspace_bytes > kWorkspaceBytes ? workspace_bytes - kWorkspaceBytes : 0;
    const PrefillPlan pl = prefill_plan(B, N, K, avail);
    return pl.est_us < cuda_core_us(B, N, K);
}

// How a grouped call runs: one CUDA-core launch over all matrices, one
// tensor-core launch whose CTAs the matrices share (small ones, such as k / v
// projections, then no longer leave SMs idle), or each matrix as its own
// logq_linear call -- whichever is estimated fastest; batches the CUDA-core
// kernel always takes stay there.  A smaller workspace can only slow the
// options that split k ranges, so the workspace the choice needs
// (part_bytes) leads to the same choice.
struct GroupChoice {
    enum { kCudaCores, kTensorCores, kSingles } kind;
    size_t part_bytes;
};

GroupChoice choose_group(int bits, int64_t B, const int64_t* N, int count, int64_t K, size_t workspace_bytes)
{
    GroupChoice ch{GroupChoice::kCudaCores, 0};
    if (!tensor_core_batch(bits, B)) return ch;
    const size_t avail = workspace_bytes > kWorkspaceBytes ? workspace_bytes - kWorkspaceBytes : 0;
    const bool cuda_ok = gemv_supports(bits, B);
    double cuda_us = 2.0, singles_us = 0.0;
    size_t single_part = 0;
    for (int i = 0; i < count; ++i) {
        const PrefillPlan pl = prefill_plan(B, N[i], K, avail);
        double us = pl.est_us;
        size_t part = pl.part_bytes;
        if (cuda_ok) {
            const double c = cuda_core_us(B, N[i], K);
            cuda_us += c - 2.0;
            if (c <= us) {
                us = c;
                part = 0;
            }
        }
        singles_us += us;
        single_part = part > single_part ? part : single_part;
    }
    const PrefillPlan gp = prefill_plan(B, N, count, K, avail);
    double best = cuda_ok ? cuda_us : 1e300;
    if (count > 1 && gp.est_us < best) {
        best = gp.est_us;
        ch = GroupChoice{GroupChoice::kTensorCores, gp.part_bytes};
    }
    if (singles_us < best)
        ch = GroupChoice{GroupChoice::kSingles, single_part};
    return ch;
}

}  // namespace

extern "C" {

logq_status logq_build_codebook(int bits, double base, double range, int flags, logq_codebook* out)
{
    if (!out || (bits != 3 && bits != 4 && bits != 8)) return LOGQ_ERR_INVALID_ARG;
    if (!isfinite(base) || !(base > 1.0) || !isfinite(range) || !(range > 0.0))
        return LOGQ_ERR_INVALID_ARG;
    if (flags != LOGQ_SHIFT_EXACT && flags != LOGQ_SHIFT_FLOOR) return LOGQ_ERR_INVALID_ARG;

    logq_codebook cb;
    memset(&cb, 0, sizeof cb);
    const int qmax = (1 << (bits - 1)) - 1;
    cb.bits = bits;
    cb.qmax = qmax;
    cb.flags = flags;
    cb.base = base;
    cb.range = range;
    // Eq. (4): s aligns w_max with q_max.  Exact mode keeps log_b(range)
    // unrounded so the top level is the range itself; floor mode is Eq. (4)
    // as printed.
    const long e_floor = (flags == LOGQ_SHIFT_FLOOR) ? floor_log_base(range, base) : 0;
    cb.shift = (flags == LOGQ_SHIFT_FLOOR) ? (double)qmax - (double)e_floor
                                           : (double)qmax - log(range) / log(base);

    // Eq. (2): L_m = b^(m - s).  Exact mode: b^(m - q_max) * range.
    double L[128] = {0};
    for (int m = 1; m <= qmax; ++m)
        L[m] = (flags == LOGQ_SHIFT_FLOOR) ? pow(base, (double)m - cb.shift)
                                           : range * pow(base, (double)(m - qmax));
    const int half = 1 << (bits - 1);
    for (int c = 0; c < 2 * half; ++c) {
        const int m = c & (half - 1);
        const float mag = (float)L[m];
        const float v = (c & half) ? -mag : mag;
        cb.level[c] = v;
        cb.level_bf16[c] = bf16_bits_of(v);
        cb.level_f16[c] = f16_bits_of(v);
    }
    // Decision boundary between L_j and L_{j+1}: round(log_b|w| + s) >= j + 1
    // exactly when |w| >= b^(j + 1/2 - s).
    for (int j = 0; j < 128; ++j) {
        if (j < qmax) {
            const double t = (flags == LOGQ_SHIFT_FLOOR)
                                 ? pow(base, (double)j + 0.5 - cb.shift)
                                 : range * pow(base, (double)j + 0.5 - (double)qmax);
            cb.thresh[j] = round_up_f32(t);
        } else {
            cb.thresh[j] = INFINITY;
        }
    }
    *out = cb;
    return LOGQ_OK;
}

size_t logq_packed_bytes(int64_t N, int64_t K, int bits)
{
    if (N <= 0 || K <= 0 || (K % 128) != 0) return 0;
    if (bits == 8) return (size_t)N * (size_t)K;
    if (bits == 4) return (size_t)N * (size_t)(K / 2);
    if (bits == 3) return (size_t)N * (size_t)(K / 32 * 12);
    return 0;
}

size_t logq_workspace_bytes(void) { return kWorkspaceBytes; }

size_t logq_linear_workspace_bytes(int64_t B, int64_t N, int64_t K, int bits)
{
    if (B <= 0 || logq_packed_bytes(N, K, bits) == 0) return 0;
    if (!tensor_core_batch(bits, B)) return kWorkspaceBytes;
    if (gemv_supports(bits, B) && !use_small_batch_tc(bits, B, N, K, (size_t)-1)) return kWorkspaceBytes;
    return kWorkspaceBytes + prefill_plan(B, N, K, (size_t)-1).part_bytes;
}

size_t logq_linear_grouped_workspace_bytes(int64_t B, const int64_t* N, int count, int64_t K, int bits)
{
    if (!N || count < 1 || count > 4 || B <= 0) return 0;
    for (int i = 0; i < count; ++i)
        if (logq_packed_bytes(N[i], K, bits) == 0) return 0;
    return kWorkspaceBytes + choose_group(bits, B, N, count, K, (size_t)-1).part_bytes;
}

logq_status logq_quantize(const float* W, int64_t N, int64_t K, int bits, double base,
                          double range, int flags, uint8_t* codes, logq_codebook* cb_out,
                          void* workspace, size_t workspace_bytes, void* stream)
{
    const logq_status st = check_quantize_args(W, N, K, bits, base, range, flags, codes);
    if (st != LOGQ_OK) return st;
    if (!workspace || !aligned16(workspace) || workspace_bytes < kWorkspaceBytes)
        return LOGQ_ERR_WORKSPACE;
    return quantize_with(W, N, K, bits, base, range, flags, codes, cb_out, static_cast<Workspace*>(workspace),
                         static_cast<cudaStream_t>(stream));
}

size_t logq_energy_scratch_bytes(void) { return sizeof(EnergyState); }

logq_status logq_quantize_energy(const float* W, int64_t N, int64_t K, int bits, double eps, int flags,
                                 uint8_t* codes, logq_codebook* cb_out, double* wmin_out,
                                 void* workspace, size_t workspace_bytes, void* scratch,
                                 size_t scratch_bytes, void* stream)
{
    if (!W || !codes || !aligned16(W) || !aligned16(codes)) return LOGQ_ERR_INVALID_ARG;
    if (logq_packed_bytes(N, K, bits) == 0) return LOGQ_ERR_INVALID_ARG;
    if (!isfinite(eps) || !(eps > 0.0) || eps > 1.0) return LOGQ_ERR_INVALID_ARG;
    if (flags != LOGQ_SHIFT_EXACT && flags != LOGQ_SHIFT_FLOOR) return LOGQ_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < kWorkspaceBytes) return LOGQ_ERR_WORKSPACE;
    if (!scratch || !aligned16(scratch) || scratch_bytes < sizeof(EnergyState)) return LOGQ_ERR_WORKSPACE;
    if (N > (int64_t(1) << 40) / K) return LOGQ_ERR_INVALID_ARG;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    Workspace* ws = static_cast<Workspace*>(workspace);
    EnergyState* st = static_cast<EnergyState*>(scratch);
    cudaError_t e = cudaMemsetAsync(ws, 0, 2 * sizeof(uint32_t), s);
    if (e != cudaSuccess) return LOGQ_ERR_CUDA;
    // Sec. 3.2: w_max and the Eq. (5) w_min, on the device
    if ((e = launch_energy_range(W, N * K, eps, st, ws, s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    uint32_t host_words[2] = {0, 0}, sel[2] = {0, 0};      // sel: w_min bits, window failure
    if ((e = cudaMemcpyAsync(host_words, ws, sizeof host_words, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
        return LOGQ_ERR_CUDA;
    if ((e = cudaMemcpyAsync(sel, &st->wmin_bits, sizeof sel, cudaMemcpyDeviceToHost, s)) != cudaSuccess)
        return LOGQ_ERR_CUDA;
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (host_words[1]) return LOGQ_ERR_NONFINITE;
    float fmax, fmin;
    memcpy(&fmax, &host_words[0], 4);
    memcpy(&fmin, &sel[0], 4);
    if (!(fmax > 0.0f)) return LOGQ_ERR_INVALID_ARG;     // all-zero weights
    if (sel[1]) return LOGQ_ERR_CUDA;                    // selection inconsistent (not expected)
    if (!(fmin > 0.0f)) return LOGQ_ERR_INVALID_ARG;
    if (!(fmin < fmax)) return LOGQ_ERR_INVALID_ARG;                      // Eq. (3) would give b = 1
    const int qmax = (1 << (bits - 1)) - 1;
    const double base = pow((double)fmax / (double)fmin, 1.0 / (double)qmax);   // Eq. (3)

    logq_codebook cb;
    logq_status st_cb = logq_build_codebook(bits, base, (double)fmax, flags, &cb);
    if (st_cb != LOGQ_OK) return st_cb;
    QuantParams p;
    memset(&p, 0, sizeof p);
    for (int j = 0; j < 128; ++j) p.thresh[j] = cb.thresh[j];
    p.qmax = cb.qmax;
    p.bits = bits;
    p.check_nonfinite = 0;          // the range pass already looked at every weight
    if ((e = launch_quantize(W, N, K, p, codes, ws, s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (cb_out) *cb_out = cb;
    if (wmin_out) *wmin_out = (double)fmin;
    return LOGQ_OK;
}

size_t logq_gptq_factor_scratch_bytes(int64_t K)
{
    if (K <= 0 || (K % 128) != 0 || K > 65536) return 0;
    return gptq_factor_scratch_bytes(K);
}

logq_status logq_gptq_factor(const float* H, int64_t K, double damp, float* U, uint8_t* dead, void* scratch,
                             size_t scratch_bytes, void* stream)
{
    if (!H || !U || !aligned16(H) || !aligned16(U)) return LOGQ_ERR_INVALID_ARG;
    if (K <= 0 || (K % 128) != 0 || K > 65536) return LOGQ_ERR_INVALID_ARG;
    if (!(damp >= 0.0) || !isfinite(damp)) return LOGQ_ERR_INVALID_ARG;
    if (!scratch || !aligned16(scratch) || scratch_bytes < gptq_factor_scratch_bytes(K)) return LOGQ_ERR_WORKSPACE;
    uint32_t not_pd = 0;
    const cudaError_t e = launch_gptq_factor(H, K, damp, U, dead, scratch, &not_pd, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_status(e);
    return not_pd ? LOGQ_ERR_NOT_PD : LOGQ_OK;
}

size_t logq_gptq_scratch_bytes(int64_t N, int64_t K)
{
    if (N <= 0 || K <= 0 || (K % 128) != 0) return 0;
    return gptq_scratch_bytes(N, K);
}

logq_status logq_gptq(const float* W, int64_t N, int64_t K, const float* U, const uint8_t* dead,
                      const logq_codebook* cb, uint8_t* codes, void* scratch, size_t scratch_bytes, void* stream)
{
    if (!W || !U || !cb || !codes) return LOGQ_ERR_INVALID_ARG;
    if (!aligned16(W) || !aligned16(U) || !aligned16(codes)) return LOGQ_ERR_INVALID_ARG;
    if (logq_packed_bytes(N, K, cb->bits) == 0) return LOGQ_ERR_INVALID_ARG;
    if (cb->qmax != (1 << (cb->bits - 1)) - 1) return LOGQ_ERR_INVALID_ARG;
    if (N > (int64_t(1) << 40) / K) return LOGQ_ERR_INVALID_ARG;
    if (cb->bits != 4 && cb->bits != 8) return LOGQ_ERR_UNSUPPORTED;
    if (!scratch || !aligned16(scratch) || scratch_bytes < gptq_scratch_bytes(N, K)) return LOGQ_ERR_WORKSPACE;
    const cudaError_t e = launch_gptq(W, N, K, U, dead, cb->bits, cb->thresh, cb->level, cb->qmax, codes, scratch,
                                      static_cast<cudaStream_t>(stream));
    return cuda_status(e);
}

logq_status logq_linear(const uint8_t* codes, const logq_codebook* cb, const void* X,
                        logq_dtype x_dtype, int64_t B, int64_t N, int64_t K, void* Y,
                        logq_dtype y_dtype, void* workspace, size_t workspace_bytes, void* stream)
{
    if (!codes || !cb || !X || !Y) return LOGQ_ERR_INVALID_ARG;
    if (!aligned16(codes) || !aligned16(X) || !aligned16(Y)) return LOGQ_ERR_INVALID_ARG;
    if (B <= 0 || logq_packed_bytes(N, K, cb->bits) == 0) return LOGQ_ERR_INVALID_ARG;
    if (cb->qmax != (1 << (cb->bits - 1)) - 1) return LOGQ_ERR_INVALID_ARG;
    if (x_dtype != LOGQ_BF16 && x_dtype != LOGQ_F16) return LOGQ_ERR_UNSUPPORTED;
    if (y_dtype != LOGQ_F32 && y_dtype != x_dtype) return LOGQ_ERR_UNSUPPORTED;
    if (N > (int64_t(1) << 31) || K > (int64_t(1) << 30) || B > (int64_t(1) << 31))
        return LOGQ_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < kWorkspaceBytes)
        return LOGQ_ERR_WORKSPACE;

    LinearArgs a;
    memset(&a, 0, sizeof a);
    a.codes = codes;
    a.X = X;
    a.Y = Y;
    a.B = B;
    a.N = N;
    a.K = K;
    a.bits = cb->bits;
    a.x_f16 = (x_dtype == LOGQ_F16);
    a.y_dtype = (int)y_dtype;
    const uint16_t* tab = a.x_f16 ? cb->level_f16 : cb->level_bf16;
    for (int c = 0; c < (1 << cb->bits); ++c) a.lvl16[c] = tab[c];
    a.ws = static_cast<Workspace*>(workspace);
    a.ws_bytes = workspace_bytes;

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (gemv_supports(cb->bits, B) && !use_small_batch_tc(cb->bits, B, N, K, workspace_bytes))
        return cuda_status(launch_gemv(a, s));
    const cudaError_t e = launch_prefill(a, s);
    if (e == cudaErrorNotSupported) return LOGQ_ERR_UNSUPPORTED;
    return cuda_status(e);
}

logq_status logq_linear_grouped(const logq_linear_item* items, int count, const void* X,
                                logq_dtype x_dtype, int64_t B, int64_t K, logq_dtype y_dtype,
                                const void* l2_prefetch, size_t l2_prefetch_bytes,
                                void* workspace, size_t workspace_bytes, void* stream)
{
    if (!items || count < 1 || count > 4 || !X || !aligned16(X)) return LOGQ_ERR_INVALID_ARG;
    if (x_dtype != LOGQ_BF16 && x_dtype != LOGQ_F16) return LOGQ_ERR_UNSUPPORTED;
    if (y_dtype != LOGQ_F32 && y_dtype != x_dtype) return LOGQ_ERR_UNSUPPORTED;
    if (B <= 0 || B > (int64_t(1) << 31) || K > (int64_t(1) << 30)) return LOGQ_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < kWorkspaceBytes) return LOGQ_ERR_WORKSPACE;
    if (l2_prefetch_bytes > 0 && !l2_prefetch) return LOGQ_ERR_INVALID_ARG;
    int bits = 0;
    for (int i = 0; i < count; ++i) {
        const logq_linear_item& it = items[i];
        if (!it.codes || !it.cb || !it.Y || !aligned16(it.codes) || !aligned16(it.Y)) return LOGQ_ERR_INVALID_ARG;
        if (it.N > (int64_t(1) << 31) || logq_packed_bytes(it.N, K, it.cb->bits) == 0) return LOGQ_ERR_INVALID_ARG;
        if (it.cb->qmax != (1 << (it.cb->bits - 1)) - 1) return LOGQ_ERR_INVALID_ARG;
        if (i == 0) bits = it.cb->bits;
        else if (it.cb->bits != bits) return LOGQ_ERR_INVALID_ARG;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    Workspace* ws = static_cast<Workspace*>(workspace);
    const int x_f16 = (x_dtype == LOGQ_F16);
    GroupArgs g;
    memset(&g, 0, sizeof g);
    g.count = count;
    for (int i = 0; i < count; ++i) {
        g.item[i].codes = items[i].codes;
        g.item[i].Y = items[i].Y;
        g.item[i].N = items[i].N;
        const uint16_t* tab = x_f16 ? items[i].cb->level_f16 : items[i].cb->level_bf16;
        for (int c = 0; c < (1 << bits); ++c) g.item[i].lvl16[c] = tab[c];
    }
    g.X = X;
    g.B = B;
    g.K = K;
    g.bits = bits;
    g.x_f16 = x_f16;
    g.y_dtype = (int)y_dtype;
    g.ws = ws;
    int64_t Ns[4];
    for (int i = 0; i < count; ++i) Ns[i] = items[i].N;
    const GroupChoice ch = choose_group(bits, B, Ns, count, K, workspace_bytes);
    if (ch.kind == GroupChoice::kCudaCores) {
        aligned_prefetch_range(l2_prefetch, l2_prefetch_bytes, &g.pf, &g.pf_bytes);
        return cuda_status(launch_gemv_group(g, s));
    }
    if (ch.kind == GroupChoice::kTensorCores) {
        const cudaError_t e = launch_prefill_group(g, workspace_bytes, s);
        if (e == cudaErrorNotSupported) return LOGQ_ERR_UNSUPPORTED;
        return cuda_status(e);
    }
    for (int i = 0; i < count; ++i) {
        const logq_status st = logq_linear(items[i].codes, items[i].cb, X, x_dtype, B, items[i].N, K, items[i].Y,
                                           y_dtype, workspace, workspace_bytes, stream);
        if (st != LOGQ_OK) return st;
    }
    return LOGQ_OK;
}

logq_status logq_workspace_status(void* workspace, void* stream, uint32_t* detail)
{
    if (!workspace || !aligned16(workspace)) return LOGQ_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    Workspace* ws = static_cast<Workspace*>(workspace);
    uint32_t words[2] = {0, 0};
    if (cudaMemcpyAsync(words, &ws->error, sizeof words, cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return LOGQ_ERR_CUDA;
    if (cudaMemsetAsync(&ws->error, 0, sizeof words, s) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return LOGQ_ERR_CUDA;
    if (detail) *detail = words[1];
    return words[0] ? LOGQ_ERR_TIMEOUT : LOGQ_OK;
}

const char* logq_status_string(logq_status status)
{
    switch (status) {
    case LOGQ_OK: return "ok";
    case LOGQ_ERR_INVALID_ARG: return "invalid argument";
    case LOGQ_ERR_NONFINITE: return "weights contain NaN or Inf";
    case LOGQ_ERR_UNSUPPORTED: return "unsupported configuration";
    case LOGQ_ERR_CUDA: return "CUDA runtime error";
    case LOGQ_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case LOGQ_ERR_TIMEOUT: return "device pipeline wait exceeded its bound";
    case LOGQ_ERR_NOT_PD: return "damped Hessian is not positive definite";
    }
    return "unknown status";
}

int logq_device_sm_count(void) { return sm_count(); }

}  // extern "C"
