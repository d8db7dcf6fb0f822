// GPTQ with the Log_b quantiser (the calibration the paper runs its
// quantiser in; GPTQ's published procedure, restated): with Hd^-1 = U^T U the
// upper Cholesky factor of the damped inverse Hessian, the columns of W are
// quantised in order; after column j the error e = (w_j - level(q_j)) / U_jj
// is compensated on every later column c by w_c -= e * U_jc.
//
// Device layout: a working copy of W (fp32, [N][K]) in the caller's scratch,
// processed in blocks of 128 columns.
//   gptq_block_kernel: one CTA per 32 rows.  The rows' 128-column slab and the
//     128 x 128 block of U sit in shared memory; column by column, 32 threads
//     quantise (boundary search, Eq. (1) as m = #{ t : |w| >= thresh[t] }) and
//     form the errors, then all threads update the rest of the slab.  The
//     slab's codes are packed at the end and its errors kept (E, [N][128]).
//   gptq_update_kernel: the columns after the block, W[:, rest] -= E U[block, rest],
//     an fp32 tiled product (64 x 64 outputs per CTA).
// The order of every sum is fixed, so a run is deterministic.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "internal.h"

namespace logq {
namespace {

constexpr int kCols = 128;         // columns per block (K is a multiple of 128)
constexpr int kRows = 32;          // rows per CTA of the block kernel
constexpr int kThreads = 256;
constexpr int kPad = kCols + 1;    // slab row stride (column reads stay bank-distinct)

struct GptqTables {
    uint32_t thresh[128];          // fp32 boundaries as bit patterns, +Inf beyond q_max - 1
    float level[128];              // fp32 levels L_0 .. L_qmax
    int32_t bits;
    int32_t qmax;
};

template <int BITS>
__global__ void __launch_bounds__(kThreads) gptq_block_kernel(float* __restrict__ Wk, int64_t N, int64_t K,
                                                              const float* __restrict__ U, int64_t j0,
                                                              const __grid_constant__ GptqTables tb,
                                                              uint8_t* __restrict__ codes, float* __restrict__ E)
{
    extern __shared__ float sm[];
    float* Ub = sm;                                   // [kCols][kCols]
    float* Wt = Ub + kCols * kCols;                   // [kRows][kPad]
    float* es = Wt + kRows * kPad;                    // [kRows]
    int8_t* qs = reinterpret_cast<int8_t*>(es + kRows);   // [kRows][kCols]
    __shared__ uint32_t th[128];
    __shared__ float lv[128];
    const int tid = threadIdx.x;
    const int64_t r0 = (int64_t)blockIdx.x * kRows;
    if (tid < 128) {
        th[tid] = tb.thresh[tid];
        lv[tid] = tb.level[tid];
    }
    for (int i = tid; i < kCols * kCols; i += kThreads) {
        const int a = i / kCols, c = i % kCols;
        Ub[i] = U[(j0 + a) * K + j0 + c];
    }
    for (int i = tid; i < kRows * kCols; i += kThreads) {
        const int r = i / kCols, c = i % kCols;
        Wt[r * kPad + c] = (r0 + r < N) ? Wk[(r0 + r) * K + j0 + c] : 0.f;
    }
    __syncthreads();
    for (int j = 0; j < kCols; ++j) {
        if (tid < kRows) {
            const float w = Wt[tid * kPad + j];
            const uint32_t u = __float_as_uint(w) & 0x7fffffffu;
            int m = 0;
#pragma unroll
            for (int step = 64; step >= 1; step >>= 1)
                if (u >= th[m + step - 1]) m += step;
            const float deq = m ? (w < 0.f ? -lv[m] : lv[m]) : 0.f;
            qs[tid * kCols + j] = (int8_t)(w < 0.f ? -m : m);
            const float e = (w - deq) / Ub[j * kCols + j];
            es[tid] = e;
            if (r0 + tid < N) E[(r0 + tid) * kCols + j] = e;
        }
        __syncthreads();
        const int rest = kCols - 1 - j;
        for (int i = tid; i < kRows * rest; i += kThreads) {
            const int r = i / rest, c = j + 1 + i % rest;
            Wt[r * kPad + c] -= es[r] * Ub[j * kCols + c];
        }
        __syncthreads();
    }
    // sign-magnitude codes of the slab (the layout of include/logq.h)
    auto code = [&](int8_t qv) -> uint32_t {
        return qv < 0 ? ((uint32_t)(-qv) | (1u << (BITS - 1))) : (uint32_t)qv;
    };
    if constexpr (BITS == 4) {
        for (int i = tid; i < kRows * (kCols / 2); i += kThreads) {
            const int r = i / (kCols / 2), b = i % (kCols / 2);
            if (r0 + r < N)
                codes[(r0 + r) * (K / 2) + j0 / 2 + b] =
                    (uint8_t)(code(qs[r * kCols + 2 * b]) | (code(qs[r * kCols + 2 * b + 1]) << 4));
        }
    } else {
        for (int i = tid; i < kRows * kCols; i += kThreads) {
            const int r = i / kCols, c = i % kCols;
            if (r0 + r < N) codes[(r0 + r) * K + j0 + c] = (uint8_t)code(qs[r * kCols + c]);
        }
    }
}

// W[:, c] -= sum_a E[:, a] U[j0 + a][c] for c >= c0 = j0 + 128: 64 x 64 outputs
// per CTA, 4 x 4 per thread, the 128 terms in chunks of 32 through shared memory.
__global__ void __launch_bounds__(kThreads) gptq_update_kernel(float* __restrict__ Wk, int64_t N, int64_t K,
                                                               const float* __restrict__ U,
                                                               const float* __restrict__ E, int64_t j0)
{
    __shared__ float Es[64][33];
    __shared__ float Us[32][64];
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    const int64_t c0 = j0 + kCols + (int64_t)blockIdx.y * 64;
    const int64_t rb = (int64_t)blockIdx.x * 64;
    float acc[4][4] = {};
    for (int a0 = 0; a0 < kCols; a0 += 32) {
        for (int i = tid; i < 64 * 32; i += kThreads) {
            const int r = i / 32, a = i % 32;
            Es[r][a] = (rb + r < N) ? E[(rb + r) * kCols + a0 + a] : 0.f;
        }
        for (int i = tid; i < 32 * 64; i += kThreads) {
            const int a = i / 64, c = i % 64;
            Us[a][c] = (c0 + c < K) ? U[(j0 + a0 + a) * K + c0 + c] : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int a = 0; a < 32; ++a) {
            float ev[4], uv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ev[i] = Es[ty + 16 * i][a];
#pragma unroll
            for (int i = 0; i < 4; ++i) uv[i] = Us[a][tx + 16 * i];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int k = 0; k < 4; ++k) acc[i][k] = fmaf(ev[i], uv[k], acc[i][k]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int64_t r = rb + ty + 16 * i;
        if (r >= N) continue;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int64_t c = c0 + tx + 16 * k;
            if (c < K) Wk[r * K + c] -= acc[i][k];
        }
    }
}

constexpr size_t kBlockSmem = sizeof(float) * (kCols * kCols + kRows * kPad + kRows) + kRows * kCols;

template <int BITS>
cudaError_t block_launch(float* Wk, int64_t N, int64_t K, const float* U, int64_t j0, const GptqTables& tb,
                         uint8_t* codes, float* E, cudaStream_t s)
{
    static int configured[64] = {0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        e = cudaFuncSetAttribute(gptq_block_kernel<BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kBlockSmem);
        if (e != cudaSuccess) return e;
        configured[dev] = 1;
    }
    const unsigned grid = (unsigned)((N + kRows - 1) / kRows);
    gptq_block_kernel<BITS><<<grid, kThreads, kBlockSmem, s>>>(Wk, N, K, U, j0, tb, codes, E);
    return cudaGetLastError();
}

}  // namespace

size_t gptq_scratch_bytes(int64_t N, int64_t K)
{
    const int64_t rows = (N + kRows - 1) / kRows * kRows;
    return (size_t)(N * K + rows * kCols) * sizeof(float);
}

cudaError_t launch_gptq(const float* W, int64_t N, int64_t K, const float* U, int bits, const float* thresh,
                        const float* level, int qmax, uint8_t* codes, void* scratch, cudaStream_t s)
{
    GptqTables tb;
    memset(&tb, 0, sizeof tb);
    for (int t = 0; t < 128; ++t) {
        float v = t < qmax ? thresh[t] : INFINITY;
        uint32_t b;
        memcpy(&b, &v, 4);
        tb.thresh[t] = b;
        tb.level[t] = t <= qmax ? level[t] : 0.f;
    }
    tb.bits = bits;
    tb.qmax = qmax;
    float* Wk = static_cast<float*>(scratch);
    float* E = Wk + N * K;
    cudaError_t e = cudaMemcpyAsync(Wk, W, sizeof(float) * (size_t)(N * K), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return e;
    for (int64_t j0 = 0; j0 < K; j0 += kCols) {
        e = bits == 8 ? block_launch<8>(Wk, N, K, U, j0, tb, codes, E, s)
                      : block_launch<4>(Wk, N, K, U, j0, tb, codes, E, s);
        if (e != cudaSuccess) return e;
        if (j0 + kCols < K) {
            const dim3 grid((unsigned)((N + 63) / 64), (unsigned)((K - j0 - kCols + 63) / 64));
            gptq_update_kernel<<<grid, kThreads, 0, s>>>(Wk, N, K, U, E, j0);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

}  // namespace logq
