// GPTQ with the Log_b quantiser (the calibration the paper runs its
// quantiser in; GPTQ's published procedure, restated).
//
// Factor: Hd = H + damp * mean(diag H) * I (a zero diagonal entry of H, an
// input that never fires, set to 1 first) and U, the upper Cholesky factor of
// Hd^-1 (Hd^-1 = U^T U).  With J the index reversal, let J Hd J = L L^T (lower
// Cholesky).  Then Hd = R R^T with R = J L J upper triangular, Hd^-1 =
// (R^-1)^T R^-1 and R^-1 is upper with a positive diagonal, so U = R^-1 =
// J L^-1 J: one Cholesky factorisation and one triangular inverse, in fp32.
//   - blocked right-looking Cholesky on 64 x 64 blocks: gptq_potrf_kernel
//     factors a diagonal block and replaces it by the inverse of its factor;
//     the panel below becomes L21 = A21 L11^-T and the trailing matrix
//     A22 -= L21 L21^T (both through gemm_kernel);
//   - the triangular inverse by doubling: with the diagonal blocks already
//     inverted, two neighbouring inverted blocks [A 0; B C] combine to
//     [A^-1 0; -C^-1 B A^-1  C^-1] (two products, batched over all pairs of a
//     level; the triangular operands skip their zero stages);
//   - U is the reversal of L^-1.
//
// Quantise: the columns of W in order; after column j the error
// e = (w_j - level(q_j)) / U_jj is compensated on every later column c by
// w_c -= e * U_jc.  A working copy of W (fp32, [N][K]) in the caller's scratch
// is processed in blocks of 128 columns:
//   gptq_block_kernel: one warp per row, lane l holding columns 4l .. 4l + 3 of
//     the row's 128-column slab in registers; the 128 x 128 block of U (zero
//     below the diagonal) in shared memory.  Column by column the warp takes
//     the column's weight from its owner lane, quantises it (Eq. (1) as
//     m = #{ t : |w| >= thresh[t] }, one ballot per 32 boundaries), forms the
//     error and updates its registers; rows never synchronise with each other.
//     The slab's codes are packed at the end and its errors kept (E, [N][128]).
//   the columns after the block, W[:, rest] -= E U[block, rest], through gemm_kernel.
// Every sum has a fixed order, so a run is deterministic.
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "internal.h"

namespace logq {
namespace {

constexpr int kCols = 128;         // columns per quantisation block (K is a multiple of 128)
constexpr int kRowsPerCta = 16;    // block kernel: one warp per row
constexpr int kBlockThreads = 32 * kRowsPerCta;
constexpr int kGT = 128;           // gemm_kernel: output tile (rows and columns)
constexpr int kGK = 32;            // gemm_kernel: terms per shared-memory stage
constexpr int kGemmThreads = 256;
constexpr int kNb = 64;            // Cholesky block
constexpr size_t kFactorState = 256;   // bytes of factor state ahead of the work matrix

struct GptqTables {
    uint32_t thresh[128];          // fp32 boundaries as bit patterns, 0xffffffff beyond q_max - 1
    float level[128];              // fp32 levels L_0 .. L_qmax
    int32_t bits;
    int32_t qmax;
};

struct FactorState {
    double mean;                   // mean of H's diagonal
    uint32_t not_pd;               // a Cholesky pivot was not positive (or not finite)
};

// C = beta C + alpha A B, A [M][Kd] row-major; B [Kd][N] row-major, or with BT
// given as [N][Kd] (C = beta C + alpha A B^T).  Batched over blockIdx.z with
// element strides sA, sB, sC.  Kd is a multiple of 32; N, the leading
// dimensions and the batch strides are multiples of 4 and the bases 16-byte
// aligned.  LOWER: tiles strictly above the diagonal are skipped.  TRI_A: A is
// lower triangular (A[m][k] = 0 for k > m), TRI_B: B is lower triangular
// (B[k][n] = 0 for k < n); the stages that hold only such zeros are skipped,
// the others read the zeros, which must be stored.
struct GemmArgs {
    const float* A;
    const float* B;
    float* C;
    int64_t M, N, Kd;
    int64_t lda, ldb, ldc;
    int64_t sA, sB, sC;
    float alpha, beta;
};

// 128 x 128 outputs per CTA; thread (tx, ty) owns rows 4ty + {0..3},
// 64 + 4ty + {0..3} and columns 4tx + {0..3}, 64 + 4tx + {0..3}; both operands
// are staged k-major in shared memory and read as float4.
template <bool BT, bool LOWER, bool TRI_A, bool TRI_B>
__global__ void __launch_bounds__(kGemmThreads, 2) gemm_kernel(const __grid_constant__ GemmArgs g)
{
    __shared__ __align__(16) float As[kGK][kGT + 4];
    __shared__ __align__(16) float Bs[kGK][kGT + 4];
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    if (LOWER && blockIdx.y > blockIdx.x) return;
    const int64_t r0 = (int64_t)blockIdx.x * kGT, c0 = (int64_t)blockIdx.y * kGT;
    const float* A = g.A + blockIdx.z * g.sA;
    const float* B = g.B + blockIdx.z * g.sB;
    float* C = g.C + blockIdx.z * g.sC;
    int64_t k_begin = 0, k_end = g.Kd;
    if (TRI_B) k_begin = c0 < g.Kd ? c0 / kGK * kGK : g.Kd;
    if (TRI_A && r0 + kGT < k_end) k_end = r0 + kGT;
    float acc[8][8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[i][k] = 0.f;
    for (int64_t k0 = k_begin; k0 < k_end; k0 += kGK) {
        for (int i = tid; i < kGT * kGK / 4; i += kGemmThreads) {
            const int rr = i / (kGK / 4), q = i % (kGK / 4);
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (r0 + rr < g.M) v = *reinterpret_cast<const float4*>(A + (r0 + rr) * g.lda + k0 + 4 * q);
            As[4 * q + 0][rr] = v.x;
            As[4 * q + 1][rr] = v.y;
            As[4 * q + 2][rr] = v.z;
            As[4 * q + 3][rr] = v.w;
        }
        if constexpr (BT) {
            for (int i = tid; i < kGT * kGK / 4; i += kGemmThreads) {
                const int nn = i / (kGK / 4), q = i % (kGK / 4);
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (c0 + nn < g.N) v = *reinterpret_cast<const float4*>(B + (c0 + nn) * g.ldb + k0 + 4 * q);
                Bs[4 * q + 0][nn] = v.x;
                Bs[4 * q + 1][nn] = v.y;
                Bs[4 * q + 2][nn] = v.z;
                Bs[4 * q + 3][nn] = v.w;
            }
        } else {
            for (int i = tid; i < kGK * kGT / 4; i += kGemmThreads) {
                const int a = i / (kGT / 4), q = i % (kGT / 4);
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (c0 + 4 * q < g.N) v = *reinterpret_cast<const float4*>(B + (k0 + a) * g.ldb + c0 + 4 * q);
                *reinterpret_cast<float4*>(&Bs[a][4 * q]) = v;
            }
        }
        __syncthreads();
#pragma unroll 4
        for (int a = 0; a < kGK; ++a) {
            const float4 e0 = *reinterpret_cast<const float4*>(&As[a][4 * ty]);
            const float4 e1 = *reinterpret_cast<const float4*>(&As[a][64 + 4 * ty]);
            const float4 u0 = *reinterpret_cast<const float4*>(&Bs[a][4 * tx]);
            const float4 u1 = *reinterpret_cast<const float4*>(&Bs[a][64 + 4 * tx]);
            const float ev[8] = {e0.x, e0.y, e0.z, e0.w, e1.x, e1.y, e1.z, e1.w};
            const float uv[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
            for (int i = 0; i < 8; ++i)
#pragma unroll
                for (int k = 0; k < 8; ++k) acc[i][k] = fmaf(ev[i], uv[k], acc[i][k]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int64_t rr = r0 + (i < 4 ? 4 * ty + i : 64 + 4 * ty + i - 4);
        if (rr >= g.M) continue;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int64_t c = c0 + 64 * h + 4 * tx;
            if (c >= g.N) continue;
            float4* p = reinterpret_cast<float4*>(C + rr * g.ldc + c);
            float4 o;
            if (g.beta == 0.f) {
                o = make_float4(g.alpha * acc[i][4 * h + 0], g.alpha * acc[i][4 * h + 1],
                                g.alpha * acc[i][4 * h + 2], g.alpha * acc[i][4 * h + 3]);
            } else {
                o = *p;
                o.x = g.beta * o.x + g.alpha * acc[i][4 * h + 0];
                o.y = g.beta * o.y + g.alpha * acc[i][4 * h + 1];
                o.z = g.beta * o.z + g.alpha * acc[i][4 * h + 2];
                o.w = g.beta * o.w + g.alpha * acc[i][4 * h + 3];
            }
            *p = o;
        }
    }
}

// mean(diag H) in fp64 (fixed order: strided partial sums, then a tree) and
// the dead-input mask.  One CTA of 1024 threads.
__global__ void __launch_bounds__(1024) gptq_diag_kernel(const float* __restrict__ H, int64_t K,
                                                         FactorState* st, uint8_t* __restrict__ dead)
{
    __shared__ double part[1024];
    const int tid = threadIdx.x;
    double s = 0.0;
    for (int64_t j = tid; j < K; j += 1024) {
        const float h = H[j * K + j];
        s += (double)h;
        if (dead) dead[j] = h == 0.f;
    }
    part[tid] = s;
    __syncthreads();
    for (int w = 512; w >= 1; w >>= 1) {
        if (tid < w) part[tid] += part[tid + w];
        __syncthreads();
    }
    if (tid == 0) {
        st->mean = part[0] / (double)K;
        st->not_pd = 0;
    }
}

// A = J Hd J (rows and columns reversed), damping on the diagonal.
__global__ void gptq_prep_kernel(const float* __restrict__ H, int64_t K, double damp, const FactorState* st,
                                 float* __restrict__ A)
{
    const double add = damp * st->mean;
    const int64_t total = K * K;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = idx / K, j = idx % K;
        const float h = H[(K - 1 - i) * K + (K - 1 - j)];
        float v = h;
        if (i == j) v = (float)((h == 0.f ? 1.0 : (double)h) + add);
        A[idx] = v;
    }
}

// Cholesky of the 64 x 64 diagonal block at (k0, k0) (lower triangle read),
// then the inverse of its factor, written back in its place with zeros above
// the diagonal.  One CTA of 256 threads: a 16 x 16 layout for the updates, four
// threads per column of the inverse.
__global__ void __launch_bounds__(256) gptq_potrf_kernel(float* __restrict__ A, int64_t K, int64_t k0,
                                                         FactorState* st)
{
    __shared__ float a[kNb][kNb + 1];
    __shared__ float inv[kNb][kNb + 1];
    const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
    for (int i = tid; i < kNb * kNb; i += 256) {
        const int r = i / kNb, c = i % kNb;
        a[r][c] = c <= r ? A[(k0 + r) * K + k0 + c] : 0.f;
    }
    __syncthreads();
    for (int j = 0; j < kNb; ++j) {
        const float p = a[j][j];
        const float d = sqrtf(p);
        if (tid == 0 && (!(p > 0.f) || !isfinite(p))) st->not_pd = 1;
        if (tid > j && tid < kNb) a[tid][j] = a[tid][j] / d;
        __syncthreads();
        if (tid == 0) a[j][j] = d;
        for (int i = j + 1 + ty; i < kNb; i += 16) {
            const float lij = a[i][j];
            for (int k = j + 1 + tx; k <= i; k += 16) a[i][k] -= lij * a[k][j];
        }
        __syncthreads();
    }
    {   // column c of the inverse by forward substitution, each sum split over four lanes
        const int c = tid / 4, q = tid % 4;
        for (int i = 0; i < kNb; ++i) {
            float part = 0.f;
            if (i > c)
                for (int k = c + q; k < i; k += 4) part = fmaf(a[i][k], inv[k][c], part);
            part += __shfl_xor_sync(0xffffffffu, part, 1);
            part += __shfl_xor_sync(0xffffffffu, part, 2);
            if (q == 0) inv[i][c] = i < c ? 0.f : ((i == c ? 1.f : 0.f) - part) / a[i][i];
            __syncwarp();
        }
    }
    __syncthreads();
    for (int i = tid; i < kNb * kNb; i += 256) {
        const int r = i / kNb, c = i % kNb;
        A[(k0 + r) * K + k0 + c] = inv[r][c];
    }
}

__global__ void gptq_zero_upper_kernel(float* __restrict__ A, int64_t K)
{
    const int64_t total = K * K;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x)
        if (idx % K > idx / K) A[idx] = 0.f;
}

// U[i][j] = Linv[K-1-i][K-1-j] (upper triangular; zeros below the diagonal).
__global__ void gptq_reverse_kernel(const float* __restrict__ Li, int64_t K, float* __restrict__ U)
{
    const int64_t total = K * K;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = idx / K, j = idx % K;
        U[idx] = j >= i ? Li[(K - 1 - i) * K + (K - 1 - j)] : 0.f;
    }
}

// Working copy of W with the dead inputs' columns zeroed.
__global__ void gptq_copy_kernel(const float4* __restrict__ W, int64_t n4, int64_t K4,
                                 const uint8_t* __restrict__ dead, float4* __restrict__ Wk)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
        float4 v = W[i];
        const int64_t c = 4 * (i % K4);
        if (dead[c + 0]) v.x = 0.f;
        if (dead[c + 1]) v.y = 0.f;
        if (dead[c + 2]) v.z = 0.f;
        if (dead[c + 3]) v.w = 0.f;
        Wk[i] = v;
    }
}

template <int BITS>
__global__ void __launch_bounds__(kBlockThreads, 2) gptq_block_kernel(float* __restrict__ Wk, int64_t N, int64_t K,
                                                                      const float* __restrict__ U, int64_t j0,
                                                                      const __grid_constant__ GptqTables tb,
                                                                      uint8_t* __restrict__ codes,
                                                                      float* __restrict__ E)
{
    constexpr int kBallots = BITS == 8 ? 4 : 1;    // 127 or 7 boundaries
    extern __shared__ float4 sm4[];
    float* Ub = reinterpret_cast<float*>(sm4);     // [kCols][kCols], upper triangle of U's block
    __shared__ float lv[128];
    const int tid = threadIdx.x, lane = tid % 32;
    const int64_t r = (int64_t)blockIdx.x * kRowsPerCta + tid / 32;
    if (tid < 128) lv[tid] = tb.level[tid];
    for (int i = tid; i < kCols * kCols / 4; i += kBlockThreads) {
        const int a = i / (kCols / 4), c = 4 * (i % (kCols / 4));
        float4 v = *reinterpret_cast<const float4*>(U + (j0 + a) * K + j0 + c);
        if (c + 0 < a) v.x = 0.f;
        if (c + 1 < a) v.y = 0.f;
        if (c + 2 < a) v.z = 0.f;
        if (c + 3 < a) v.w = 0.f;
        sm4[i] = v;
    }
    uint32_t th[kBallots];
#pragma unroll
    for (int b = 0; b < kBallots; ++b) th[b] = tb.thresh[lane + 32 * b];
    __syncthreads();
    if (r >= N) return;
    const float4 w4 = *reinterpret_cast<const float4*>(Wk + r * K + j0 + 4 * lane);
    float wv[4] = {w4.x, w4.y, w4.z, w4.w};
    int qv[4] = {0, 0, 0, 0};
    float ev[4] = {0.f, 0.f, 0.f, 0.f};
    for (int j4 = 0; j4 < kCols / 4; ++j4) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int j = 4 * j4 + k;
            const float w = __shfl_sync(0xffffffffu, wv[k], j4);
            const uint32_t u = __float_as_uint(w) & 0x7fffffffu;
            int m = 0;
#pragma unroll
            for (int b = 0; b < kBallots; ++b) m += __popc(__ballot_sync(0xffffffffu, u >= th[b]));
            const float deq = m ? (w < 0.f ? -lv[m] : lv[m]) : 0.f;
            const float e = (w - deq) / Ub[j * kCols + j];
            if (lane == j4) {
                qv[k] = w < 0.f ? -m : m;
                ev[k] = e;
            }
            const float4 u4 = sm4[(j * kCols) / 4 + lane];
            wv[0] -= e * u4.x;
            wv[1] -= e * u4.y;
            wv[2] -= e * u4.z;
            wv[3] -= e * u4.w;
        }
    }
    *reinterpret_cast<float4*>(E + r * kCols + 4 * lane) = make_float4(ev[0], ev[1], ev[2], ev[3]);
    // sign-magnitude codes (the layout of include/logq.h)
    uint32_t c[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
        c[k] = qv[k] < 0 ? ((uint32_t)(-qv[k]) | (1u << (BITS - 1))) : (uint32_t)qv[k];
    if constexpr (BITS == 4)
        *reinterpret_cast<uint16_t*>(codes + r * (K / 2) + j0 / 2 + 2 * lane) =
            (uint16_t)(c[0] | (c[1] << 4) | (c[2] << 8) | (c[3] << 12));
    else
        *reinterpret_cast<uint32_t*>(codes + r * K + j0 + 4 * lane) = c[0] | (c[1] << 8) | (c[2] << 16) | (c[3] << 24);
}

constexpr size_t kBlockSmem = sizeof(float) * kCols * kCols;

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
    const unsigned grid = (unsigned)((N + kRowsPerCta - 1) / kRowsPerCta);
    gptq_block_kernel<BITS><<<grid, kBlockThreads, kBlockSmem, s>>>(Wk, N, K, U, j0, tb, codes, E);
    return cudaGetLastError();
}

template <bool BT, bool LOWER, bool TRI_A, bool TRI_B>
cudaError_t gemm(const GemmArgs& g, int64_t batch, cudaStream_t s)
{
    if (g.M <= 0 || g.N <= 0 || batch <= 0) return cudaSuccess;
    const dim3 grid((unsigned)((g.M + kGT - 1) / kGT), (unsigned)((g.N + kGT - 1) / kGT), (unsigned)batch);
    gemm_kernel<BT, LOWER, TRI_A, TRI_B><<<grid, kGemmThreads, 0, s>>>(g);
    return cudaGetLastError();
}

GemmArgs gemm_args(const float* A, int64_t lda, const float* B, int64_t ldb, float* C, int64_t ldc, int64_t M,
                   int64_t N, int64_t Kd, float alpha, float beta)
{
    GemmArgs g;
    memset(&g, 0, sizeof g);
    g.A = A;
    g.B = B;
    g.C = C;
    g.M = M;
    g.N = N;
    g.Kd = Kd;
    g.lda = lda;
    g.ldb = ldb;
    g.ldc = ldc;
    g.alpha = alpha;
    g.beta = beta;
    return g;
}

unsigned elementwise_grid(int64_t n)
{
    const int64_t b = (n + 255) / 256;
    return (unsigned)(b < 4096 ? (b > 0 ? b : 1) : 4096);
}

// Two neighbouring inverted diagonal blocks -> their combined inverse, for the
// pairs p = p0 .. p0 + count - 1 of one level (top block at p s, `half` rows;
// bottom block of c rows below it).
cudaError_t combine_pairs(float* Lw, int64_t K, int64_t s_, int64_t half, int64_t c, int64_t p0, int64_t count,
                          float* X, cudaStream_t st)
{
    const int64_t t0 = p0 * s_, b0 = t0 + half;
    // X_p = B_p A_p^-1 (A_p^-1 lower triangular)
    GemmArgs g = gemm_args(Lw + b0 * K + t0, K, Lw + t0 * K + t0, K, X, half, c, half, half, 1.f, 0.f);
    g.sA = s_ * K + s_;
    g.sB = s_ * K + s_;
    g.sC = c * half;
    cudaError_t e = gemm<false, false, false, true>(g, count, st);
    if (e != cudaSuccess) return e;
    // block (bottom, top) = -C_p^-1 X_p (C_p^-1 lower triangular)
    g = gemm_args(Lw + b0 * K + b0, K, X, half, Lw + b0 * K + t0, K, c, half, c, -1.f, 0.f);
    g.sA = s_ * K + s_;
    g.sB = c * half;
    g.sC = s_ * K + s_;
    return gemm<false, false, true, false>(g, count, st);
}

}  // namespace

size_t gptq_factor_scratch_bytes(int64_t K)
{
    return kFactorState + (size_t)(K * K + K * K / 4) * sizeof(float);
}

cudaError_t launch_gptq_factor(const float* H, int64_t K, double damp, float* U, uint8_t* dead, void* scratch,
                               uint32_t* not_pd, cudaStream_t s)
{
    FactorState* st = static_cast<FactorState*>(scratch);
    float* Lw = reinterpret_cast<float*>(static_cast<char*>(scratch) + kFactorState);
    float* X = Lw + K * K;
    gptq_diag_kernel<<<1, 1024, 0, s>>>(H, K, st, dead);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    gptq_prep_kernel<<<elementwise_grid(K * K), 256, 0, s>>>(H, K, damp, st, Lw);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // Cholesky of J Hd J; diagonal blocks end up inverted
    for (int64_t k0 = 0; k0 < K; k0 += kNb) {
        gptq_potrf_kernel<<<1, 256, 0, s>>>(Lw, K, k0, st);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        const int64_t k1 = k0 + kNb, m = K - k1;
        if (m <= 0) break;
        // L21 = A21 L11^-T, in place
        e = gemm<true, false, false, false>(
            gemm_args(Lw + k1 * K + k0, K, Lw + k0 * K + k0, K, Lw + k1 * K + k0, K, m, kNb, kNb, 1.f, 0.f), 1, s);
        if (e != cudaSuccess) return e;
        // A22 -= L21 L21^T (lower triangle)
        e = gemm<true, true, false, false>(
            gemm_args(Lw + k1 * K + k0, K, Lw + k1 * K + k0, K, Lw + k1 * K + k1, K, m, m, kNb, -1.f, 1.f), 1, s);
        if (e != cudaSuccess) return e;
    }
    gptq_zero_upper_kernel<<<elementwise_grid(K * K), 256, 0, s>>>(Lw, K);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // triangular inverse by doubling
    for (int64_t half = kNb; half < K; half *= 2) {
        const int64_t s_ = 2 * half;
        const int64_t full = K / s_;                    // pairs whose bottom block is complete
        if (full > 0 && (e = combine_pairs(Lw, K, s_, half, half, 0, full, X, s)) != cudaSuccess) return e;
        const int64_t b0 = full * s_ + half;           // a last pair with a shorter bottom block
        if (b0 < K && (e = combine_pairs(Lw, K, s_, half, K - b0, full, 1, X + full * half * half, s)) != cudaSuccess)
            return e;
    }
    gptq_reverse_kernel<<<elementwise_grid(K * K), 256, 0, s>>>(Lw, K, U);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (not_pd) {
        e = cudaMemcpyAsync(not_pd, &st->not_pd, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) return e;
        e = cudaStreamSynchronize(s);
    }
    return e;
}

size_t gptq_scratch_bytes(int64_t N, int64_t K)
{
    return (size_t)(N * K + N * kCols) * sizeof(float);
}

cudaError_t launch_gptq(const float* W, int64_t N, int64_t K, const float* U, const uint8_t* dead, int bits,
                        const float* thresh, const float* level, int qmax, uint8_t* codes, void* scratch,
                        cudaStream_t s)
{
    GptqTables tb;
    memset(&tb, 0, sizeof tb);
    for (int t = 0; t < 128; ++t) {
        uint32_t b = 0xffffffffu;              // above every |w| bit pattern: m never exceeds q_max
        if (t < qmax) memcpy(&b, &thresh[t], 4);
        tb.thresh[t] = b;
        tb.level[t] = t <= qmax ? level[t] : 0.f;
    }
    tb.bits = bits;
    tb.qmax = qmax;
    float* Wk = static_cast<float*>(scratch);
    float* E = Wk + N * K;
    cudaError_t e;
    if (dead) {
        const int64_t n4 = N * K / 4;
        gptq_copy_kernel<<<elementwise_grid(n4), 256, 0, s>>>(reinterpret_cast<const float4*>(W), n4, K / 4, dead,
                                                             reinterpret_cast<float4*>(Wk));
        e = cudaGetLastError();
    } else {
        e = cudaMemcpyAsync(Wk, W, sizeof(float) * (size_t)(N * K), cudaMemcpyDeviceToDevice, s);
    }
    if (e != cudaSuccess) return e;
    for (int64_t j0 = 0; j0 < K; j0 += kCols) {
        e = bits == 8 ? block_launch<8>(Wk, N, K, U, j0, tb, codes, E, s)
                      : block_launch<4>(Wk, N, K, U, j0, tb, codes, E, s);
        if (e != cudaSuccess) return e;
        const int64_t c1 = j0 + kCols;
        if (c1 < K) {   // W[:, c1:] -= E U[j0:c1, c1:]
            e = gemm<false, false, false, false>(
                gemm_args(E, kCols, U + j0 * K + c1, K, Wk + c1, K, N, K - c1, kCols, -1.f, 1.f), 1, s);
            if (e != cudaSuccess) return e;
        }
    }
    return cudaSuccess;
}

}  // namespace logq
