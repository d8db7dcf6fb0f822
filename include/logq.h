/*
 * logq.h -- C ABI of the GB300 (sm_103a) Log_bQuant inference library.
 *
 * Log_bQuant stores each weight of a matrix as a sign + log-level code and
 * decodes it through one codebook per matrix (paper Sec. 3.1):
 *
 *   Eq. (1)  Quant(b, s, x)   = 0 if x = 0, else sign(x) * round_clamp(log_b|x| + s)
 *   Eq. (2)  Dequant(b, s, q) = 0 if q = 0, else sign(q) * b^(|q| - s)
 *   q_max = 2^(n-1) - 1 for an n-bit code; Eq. (4) aligns w_max with q_max.
 *
 * Inference multiplies activations with the dequantised weights through a
 * lookup table (Sec. 3.3).  This library provides the steps of that path as
 * device kernels behind plain C calls:
 *   logq_build_codebook  host: (bits, base, range) -> levels and boundaries
 *   logq_quantize        device: fp32 W[N][K] -> packed codes + codebook
 *   logq_quantize_energy device: the same with w_min / w_max / b derived from W
 *                        (Sec. 3.2, Eqs. (3)-(5))
 *   logq_gptq_factor,    device: GPTQ calibration with the Log_b quantiser
 *   logq_gptq            (the paper's post-training calibration): Hessian ->
 *                        inverse-Hessian factor, then W -> packed codes
 *   logq_linear          device: codes, codebook, X[B][K] -> Y[B][N] = X * What^T
 *   logq_linear_grouped  the same for up to four matrices sharing X, one launch
 *
 * Conventions shared by every call:
 *   - Matrices are row-major and contiguous.  W and What are [N][K]
 *     (PyTorch nn.Linear layout: out x in, K contiguous); X is [B][K];
 *     Y is [B][N].
 *   - "device" pointers are CUDA global-memory addresses on the current
 *     device; "host" pointers are ordinary CPU memory.  The caller owns every
 *     buffer; the library allocates no memory and keeps no per-call state.
 *   - stream is a cudaStream_t passed as void*; NULL means the legacy default
 *     stream.  Work is enqueued on that stream in order; calls return once it
 *     is enqueued unless stated otherwise.
 *   - Every argument is validated before anything is enqueued.  A call that
 *     returns an error other than LOGQ_ERR_CUDA / LOGQ_ERR_NONFINITE has
 *     touched no device memory.
 *   - Decode launches (logq_linear with small B, logq_linear_grouped) use
 *     programmatic dependent launch: they may start while the preceding kernel
 *     on the stream finishes.  They read X and write Y only after that kernel
 *     has completed and its writes are visible, but they read the packed codes
 *     earlier, before that guarantee holds.  So the codes must be complete
 *     before the call is enqueued, ordered by a host synchronisation after the
 *     kernel that wrote them (of its stream, of an event recorded after it, or
 *     of the device), not by stream order alone.  logq_quantize and
 *     logq_quantize_energy end with such a synchronisation; after logq_gptq
 *     the caller synchronises.  Weights quantised once and reused (the decode
 *     case) meet this.
 *   - Device code never traps.  Conditions found on the device (non-finite
 *     weights, a pipeline wait that exceeded its bound) are written to the
 *     caller's workspace and reported by logq_quantize or logq_workspace_status.
 */
#ifndef LOGQ_H
#define LOGQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LOGQ_OK = 0,
    LOGQ_ERR_INVALID_ARG = 1,   /* a size, pointer, alignment or parameter is invalid */
    LOGQ_ERR_NONFINITE = 2,     /* W holds NaN or +-Inf */
    LOGQ_ERR_UNSUPPORTED = 3,   /* valid request the library does not implement */
    LOGQ_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed */
    LOGQ_ERR_WORKSPACE = 5,     /* workspace missing, too small or misaligned */
    LOGQ_ERR_TIMEOUT = 6,       /* a device-side pipeline wait hit its bound */
    LOGQ_ERR_NOT_PD = 7         /* logq_gptq_factor: the damped Hessian is not positive definite */
} logq_status;

typedef enum {
    LOGQ_F32 = 0,
    LOGQ_BF16 = 1,
    LOGQ_F16 = 2
} logq_dtype;

/* flags of logq_build_codebook / logq_quantize */
#define LOGQ_SHIFT_EXACT 0   /* s = q_max - log_b(range): the top level equals range (default) */
#define LOGQ_SHIFT_FLOOR 1   /* s = q_max - floor(log_b range), Eq. (4) as printed */

/*
 * Codebook of one weight matrix (Sec. 3.1).  Plain data: the caller owns it
 * and passes it by pointer; the library copies what it needs into kernel
 * parameters.  Entries are indexed by the n-bit code c = sign << (n-1) | m:
 *   level[m]               = +L_m,  level[2^(n-1) + m] = -L_m,
 *   L_0 = 0 (level[2^(n-1)] = -0.0f), L_m = b^(m - s) for m = 1..q_max,
 *   all rounded to nearest-even fp32 from an fp64 evaluation.
 *   thresh[j] (j < q_max) is the decision boundary tau_j = b^(j + 1/2 - s)
 *   between L_j and L_{j+1}, rounded UP to fp32, so that for an fp32 weight
 *   |w| >= thresh[j] exactly when |w| >= tau_j.  Unused entries are +Inf.
 *   level_bf16 / level_f16 are level[] rounded to nearest-even bf16 / fp16
 *   (bit patterns); logq_linear multiplies with the table of X's dtype.
 */
typedef struct logq_codebook {
    int32_t bits;            /* n: 3, 4 or 8 */
    int32_t qmax;            /* 2^(n-1) - 1 */
    int32_t flags;           /* LOGQ_SHIFT_* used */
    int32_t _pad;
    double base;             /* b */
    double shift;            /* s */
    double range;            /* w_max the codebook was built for */
    float level[256];        /* entries 0 .. 2^n - 1 used */
    float thresh[128];       /* entries 0 .. q_max - 1 used */
    uint16_t level_bf16[256];
    uint16_t level_f16[256];
} logq_codebook;

/*
 * Packed code layout (produced by logq_quantize, consumed by logq_linear):
 *   code of a weight: c = sign << (n-1) | m with m in 0..q_max and sign = 1
 *   only for negative weights with m > 0.
 *   n = 4: [N][K/2] bytes; byte j of a row holds k = 2j in bits 0-3 and
 *          k = 2j+1 in bits 4-7.
 *   n = 8: [N][K] bytes, one code per byte (sign in bit 7).
 *   n = 3: [N][3K/8] bytes; each run of 32 k is a 12-byte group of three
 *          little-endian uint32 W0, W1, W2.  Pair p (k = 2p, 2p+1 of the group)
 *          is the 6-bit field f_p = c(2p) | c(2p+1) << 3; for p = 5i + j
 *          (i < 3, j < 5) f_p is bits [6j, 6j+6) of W_i; f_15 is split two
 *          bits per word into bits 30-31 of W0 (f bits 0-1), W1 (2-3), W2 (4-5).
 * K must be a positive multiple of 128 (rows stay 16-byte aligned).
 */

/* Fill *out for an n-bit codebook with base b = base > 1 and range > 0
 * (Eq. (2) levels, Eq. (4) shift per flags).  Host only, no CUDA call.
 * Errors: LOGQ_ERR_INVALID_ARG for bits not in {3,4,8}, base <= 1 or not
 * finite, range <= 0 or not finite, unknown flags, out == NULL. */
logq_status logq_build_codebook(int bits, double base, double range, int flags,
                                logq_codebook* out);

/* Bytes of packed codes for an N x K matrix at n bits (N*K/2, N*3K/8 or N*K);
 * 0 when N <= 0, K is not a positive multiple of 128 or bits not in {3,4,8}. */
size_t logq_packed_bytes(int64_t N, int64_t K, int bits);

/* Bytes of device workspace that logq_quantize and logq_linear need (a small
 * constant).  The caller allocates it (16-byte aligned), zero-fills it once,
 * and may reuse it across calls on the same stream; calls that run at the
 * same time on different streams need separate workspaces. */
size_t logq_workspace_bytes(void);

/* Bytes of workspace with which logq_linear (and logq_linear_grouped, per
 * matrix) runs a B x N x K product at full speed: logq_workspace_bytes() plus,
 * for products that run on the tensor cores, room for fp32 partial sums when
 * the output tiles are too few to fill the GPU and each tile's k range is split
 * over several CTAs (Y is then their fixed-order sum, a second kernel on the
 * same stream).  A smaller workspace (at least logq_workspace_bytes()) is
 * accepted: the call then splits less, or, for 4-bit batches of 8..16, keeps
 * the CUDA-core kernel.  0 for invalid sizes. */
size_t logq_linear_workspace_bytes(int64_t B, int64_t N, int64_t K, int bits);

/*
 * Quantise fp32 weights W[N][K] (device) to packed codes (device) with a
 * codebook built for (bits, base, range, flags) -- Eq. (1) with the
 * decision boundaries of logq_codebook: m = #{ j : |w| >= thresh[j] }.
 *   range > 0: use it as w_max.  range <= 0: w_max = max|W| (Sec. 3.2),
 *     computed on the device; one 8-byte device-to-host read follows.
 *   cb_out (host, may be NULL) receives the codebook used.
 *   codes must hold logq_packed_bytes(N, K, bits) bytes, 16-byte aligned;
 *   W must be 16-byte aligned.
 * Synchronises `stream` once before returning (to report non-finite weights).
 * Errors: LOGQ_ERR_INVALID_ARG (sizes, pointers, alignment, codebook
 * parameters), LOGQ_ERR_WORKSPACE, LOGQ_ERR_NONFINITE (W holds NaN/Inf; codes
 * are then unspecified), LOGQ_ERR_CUDA. */
logq_status logq_quantize(const float* W, int64_t N, int64_t K, int bits, double base,
                          double range, int flags, uint8_t* codes, logq_codebook* cb_out,
                          void* workspace, size_t workspace_bytes, void* stream);

/*
 * Y[B][N] = X[B][K] * What^T with What[n][k] = table[code(n, k)] (Sec. 3.3),
 * accumulated in fp32.  table is cb->level_bf16 when x_dtype = LOGQ_BF16 and
 * cb->level_f16 when x_dtype = LOGQ_F16.
 *   codes (device): packed as above for cb->bits.  X (device): x_dtype.
 *   Y (device): y_dtype in {LOGQ_F32, x_dtype}; a 16-bit Y is the fp32 sum
 *   rounded to nearest-even.  All device pointers 16-byte aligned.
 *   B <= 16 (4-bit) or B <= 4 (3- and 8-bit) runs the decode GEMV /
 *   skinny-GEMM kernel on CUDA cores; larger B runs the prefill GEMM kernel
 *   on the tensor cores (tcgen05), as do 4-bit batches of 8..16 when the
 *   workspace (see logq_linear_workspace_bytes) lets that launch keep at
 *   least half of the SMs busy.  Calls sharing a workspace must be ordered
 *   on one stream (partial sums may live in it).
 * Asynchronous.  Errors: LOGQ_ERR_INVALID_ARG, LOGQ_ERR_UNSUPPORTED,
 * LOGQ_ERR_WORKSPACE, LOGQ_ERR_CUDA (launch).  A device-side wait that hit
 * its bound is reported later by logq_workspace_status. */
logq_status logq_linear(const uint8_t* codes, const logq_codebook* cb, const void* X,
                        logq_dtype x_dtype, int64_t B, int64_t N, int64_t K, void* Y,
                        logq_dtype y_dtype, void* workspace, size_t workspace_bytes,
                        void* stream);

/*
 * Allocation-free variant of logq_quantize (the paper has no counterpart; it
 * serves callers of this library that must not allocate device memory, such as
 * a plugin whose host application owns all device memory through its own pool,
 * or a latency-critical path that cannot take the device synchronisation an
 * allocation implies -- and that therefore cannot supply a workspace).
 * Instead of a caller workspace it uses a 256-byte scratch record kept in a
 * static device array of the library; each GPU that loads the library holds
 * that array until the process exits.  The scratch does not grow with N or K,
 * so the call accepts every size logq_quantize accepts (LOGQ_ERR_WORKSPACE would
 * report a scratch need beyond the array).  It calls no cudaMalloc, cudaFree
 * or other allocating routine.  Its first call on a device (and the first call
 * after the device's context has been replaced, e.g. by cudaDeviceReset) looks
 * up the array's device address with that device current.  All calls share
 * the one array, which keeps the last call's contents (each call clears the
 * words it needs): calls that overlap on the GPU race and must be serialised
 * by the caller.  Like
 * logq_quantize it synchronises `stream` before returning; arguments and
 * errors are those of logq_quantize, and the quantisation is the same code.
 */
logq_status logq_quantize_noalloc(const float* W, int64_t N, int64_t K, int bits, double base,
                                  double range, int flags, uint8_t* codes,
                                  logq_codebook* cb_out, void* stream);

/* Bytes of device scratch that logq_quantize_energy needs (a constant, about
 * 65 KB).  Caller-allocated, 16-byte aligned; its contents need no
 * initialisation and are overwritten by every call. */
size_t logq_energy_scratch_bytes(void);

/*
 * Self-calibrating quantisation (Sec. 3.2): derive the effective range of
 * W[N][K] (device, fp32) from the weights and quantise with it.
 *   w_max = max_i |w_i|;
 *   w_min = min { t : sum_{|w_i| <= t} w_i^2 / sum_i w_i^2 >= eps }   (Eq. (5)),
 *           the smallest weight magnitude at which the discarded energy share
 *           reaches eps (the paper uses eps = 4e-3 at 4 bits); it is always
 *           one of the |w_i|;
 *   b     = (w_max / w_min)^(1 / q_max)                                (Eq. (3));
 *   then the codebook (bits, b, w_max, flags) -- flags LOGQ_SHIFT_FLOOR is
 *   Eq. (4) as printed -- and the codes exactly as logq_quantize with those
 *   arguments would produce them.
 * The selection runs on the device in three streaming passes over W (a radix
 * selection over the bit patterns of |w|) plus the quantisation pass; energies of equal-exponent buckets are summed exactly in
 * integers and accumulated across buckets in fp64, in ascending order of |w|.
 *   eps in (0, 1].  wmin_out (host, may be NULL) receives w_min; cb_out (host,
 *   may be NULL) the codebook (its base is b, its range w_max).
 *   scratch: logq_energy_scratch_bytes() bytes of device memory.
 * Synchronises `stream` once after the range is known and once before
 * returning.
 * Errors: those of logq_quantize; LOGQ_ERR_INVALID_ARG also when eps is not in
 * (0, 1], W is all zero, or w_min == w_max (a single magnitude holds the
 * required energy, so Eq. (3) gives b = 1: no logarithmic codebook exists);
 * LOGQ_ERR_WORKSPACE also for a missing, small or misaligned scratch.
 */
logq_status logq_quantize_energy(const float* W, int64_t N, int64_t K, int bits, double eps, int flags,
                                 uint8_t* codes, logq_codebook* cb_out, double* wmin_out,
                                 void* workspace, size_t workspace_bytes, void* scratch,
                                 size_t scratch_bytes, void* stream);

/* Bytes of device scratch logq_gptq_factor needs for a K x K Hessian (1.25 K^2
 * floats and 256 bytes); 0 for invalid K. */
size_t logq_gptq_factor_scratch_bytes(int64_t K);

/*
 * The factor GPTQ compensates with (GPTQ's published procedure, the
 * calibration the paper quantises its models with, Sec. 3.3 / Sec. 4):
 * Hd = H + damp * mean(diag H) * I, a zero diagonal entry of H (an input that
 * never fires) set to 1 first; U = the upper Cholesky factor of Hd^-1
 * (Hd^-1 = U^T U), computed in fp32 on the device as the inverse of the
 * index-reversed Cholesky factor of Hd.
 *   H (device, fp32, [K][K] row-major, symmetric, 16-byte aligned): e.g.
 *     2 X^T X of the layer's calibration inputs; K a multiple of 128, at most
 *     65536.  Not modified.
 *   damp: finite, >= 0 (GPTQ's usual value is 0.01).
 *   U (device, fp32, [K][K], 16-byte aligned): receives the factor, zeros
 *     below the diagonal.
 *   dead (device, K bytes, may be NULL): receives 1 for every input whose
 *     Hessian diagonal is zero, else 0 -- hand it to logq_gptq.
 *   scratch: logq_gptq_factor_scratch_bytes(K) bytes of device memory.
 * Synchronises `stream` once (to read the positive-definiteness flag).
 * Errors: LOGQ_ERR_INVALID_ARG (sizes, pointers, alignment, damp),
 * LOGQ_ERR_WORKSPACE (scratch), LOGQ_ERR_NOT_PD (a Cholesky pivot was not
 * positive or not finite: U is then unspecified), LOGQ_ERR_CUDA.
 */
logq_status logq_gptq_factor(const float* H, int64_t K, double damp, float* U, uint8_t* dead, void* scratch,
                             size_t scratch_bytes, void* stream);

/* Bytes of device scratch logq_gptq needs for an N x K matrix (the working copy
 * of W plus the errors of one 128-column block); 0 for invalid sizes. */
size_t logq_gptq_scratch_bytes(int64_t N, int64_t K);

/*
 * GPTQ with the Log_b quantiser: the post-training calibration the paper
 * quantises its models with (Sec. 3.3 / Sec. 4, GPTQ's published procedure).
 * The columns of W are quantised in order with the codebook cb (Eq. (1) as
 * m = #{ j : |w| >= thresh[j] }); after column j the error
 * e = (w_j - level(q_j)) / U[j][j] (level = the fp32 level of the code) is
 * compensated on every later column c: w_c -= e * U[j][c].  Processed in
 * blocks of 128 columns; the columns after a block receive the block's
 * compensation as one product.
 *   W (device, fp32, [N][K], 16-byte aligned, finite): not modified; a
 *     non-finite weight gives unspecified (in-range) codes.
 *   U (device, fp32, [K][K] row-major, 16-byte aligned): the factor from
 *     logq_gptq_factor (any upper Cholesky factor of a damped inverse Hessian;
 *     its strictly lower triangle is ignored).
 *   dead (device, K bytes, may be NULL): inputs marked 1 have their weights
 *     zeroed before quantisation (they never see input), as logq_gptq_factor
 *     reports them.
 *   cb (host): the codebook (bits 4 or 8), e.g. from logq_build_codebook with
 *     the range and base of the original W.
 *   codes (device): logq_packed_bytes(N, K, bits) bytes, the packed result.
 *   scratch: logq_gptq_scratch_bytes(N, K) bytes of device memory.
 * Asynchronous (a device copy and 2 K / 128 - 1 launches on `stream`).
 * Errors: LOGQ_ERR_INVALID_ARG (sizes, pointers, alignment, codebook),
 * LOGQ_ERR_UNSUPPORTED (3-bit codebooks), LOGQ_ERR_WORKSPACE (scratch),
 * LOGQ_ERR_CUDA.
 */
logq_status logq_gptq(const float* W, int64_t N, int64_t K, const float* U, const uint8_t* dead,
                      const logq_codebook* cb, uint8_t* codes, void* scratch, size_t scratch_bytes, void* stream);

/* One matrix of logq_linear_grouped. */
typedef struct logq_linear_item {
    const uint8_t* codes;       /* device: packed codes of this matrix, N rows */
    const logq_codebook* cb;    /* host: its codebook */
    int64_t N;                  /* rows of the matrix = outputs per batch row */
    void* Y;                    /* device: output [B][N] in y_dtype */
} logq_linear_item;

/*
 * Several quantised linear layers that read the same activations X[B][K] --
 * e.g. the q/k/v or the gate/up projections of a transformer layer -- each
 * with its own per-tensor codebook (Sec. 3.1) and output: Y_i = X * What_i^T
 * (Sec. 3.3), in one call.  count is 1..4 and all items share the code width
 * of their codebooks.  With B <= 16 (4-bit) or B <= 4 (3-, 8-bit) the matrices
 * share a single decode-GEMV launch.  Larger B (and 4-bit batches of 8..16
 * that logq_linear would send to the tensor cores) runs one prefill launch
 * whose CTAs are divided among the matrices in proportion to their tiles,
 * when its estimate beats one launch per matrix (small matrices such as k / v
 * projections then share the GPU with a larger one); otherwise one launch
 * each, as logq_linear.  The workspace holds the partial sums of split k
 * ranges as for logq_linear: logq_linear_grouped_workspace_bytes gives the
 * size with which the planned launches split fully.
 * l2_prefetch (device, may be NULL) / l2_prefetch_bytes name a range the
 * call asks the L2 cache to fetch while it runs -- for a decode step, the
 * codes of the next layer -- a hint only: it is never read by the
 * computation and may be any readable device memory at any alignment (the
 * library prefetches the 16-byte aligned part inside it: the start rounded up
 * and the length down to whole 16-byte units).  A decode-GEMV launch ignores
 * a range of 20 MiB or more: codes that large stream at full rate when their
 * own launch reads them, and prefetching them would slow this one.  Asynchronous; errors
 * as logq_linear (LOGQ_ERR_INVALID_ARG also for count outside 1..4 or items
 * of different code widths).
 */
logq_status logq_linear_grouped(const logq_linear_item* items, int count, const void* X,
                                logq_dtype x_dtype, int64_t B, int64_t K, logq_dtype y_dtype,
                                const void* l2_prefetch, size_t l2_prefetch_bytes,
                                void* workspace, size_t workspace_bytes, void* stream);

/* Workspace bytes with which logq_linear_grouped of count (1..4) matrices of
 * N[0..count-1] rows (host array), code width bits and batch B runs as
 * planned: logq_workspace_bytes() plus the largest partial-sum space among
 * its launches.  A smaller workspace (at least logq_workspace_bytes()) is
 * accepted and only reduces the splits.  0 for invalid sizes. */
size_t logq_linear_grouped_workspace_bytes(int64_t B, const int64_t* N, int count, int64_t K, int bits);

/* Synchronise `stream`, read the device error word of `workspace`, clear it,
 * and return LOGQ_OK or LOGQ_ERR_TIMEOUT.  *detail (host, may be NULL)
 * receives an implementation code naming the wait that gave up. */
logq_status logq_workspace_status(void* workspace, void* stream, uint32_t* detail);

/* Static description of a status code. */
const char* logq_status_string(logq_status status);

/* Number of streaming multiprocessors of the current device (0 on error);
 * the persistent kernels size their grids from it. */
int logq_device_sm_count(void);

#ifdef __cplusplus
}
#endif

#endif /* LOGQ_H */
