// absmax reduction and quantise + pack kernels (paper Eq. (1), Sec. 3.2 w_max).
//
// Both kernels stream fp32 W once with 16-byte loads that bypass L1.
// The quantiser assigns m = #{ j : |w| >= thresh[j] } against the fp32
// decision boundaries of the codebook (rounded up from fp64), which for fp32
// weights equals round(log_b|w| + s) clamped to [0, q_max].
#include <stdint.h>

#include "internal.h"

namespace logq {
namespace {

__device__ __forceinline__ float4 ld_stream(const float4* p)
{
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void absmax_acc(float x, uint32_t& mx, uint32_t& bad)
{
    const uint32_t a = __float_as_uint(x) & 0x7fffffffu;
    const bool nf = a >= 0x7f800000u;
    bad |= nf ? 1u : 0u;
    mx = max(mx, nf ? 0u : a);   // non-negative floats order like their bit patterns
}

__global__ void __launch_bounds__(256) absmax_kernel(const float4* __restrict__ W, int64_t n4,
                                                     Workspace* ws)
{
    uint32_t mx = 0, bad = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (; i + 3 * stride < n4; i += 4 * stride) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = ld_stream(W + i + u * stride);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            absmax_acc(v[u].x, mx, bad);
            absmax_acc(v[u].y, mx, bad);
            absmax_acc(v[u].z, mx, bad);
            absmax_acc(v[u].w, mx, bad);
        }
    }
    for (; i < n4; i += stride) {
        const float4 v = ld_stream(W + i);
        absmax_acc(v.x, mx, bad);
        absmax_acc(v.y, mx, bad);
        absmax_acc(v.z, mx, bad);
        absmax_acc(v.w, mx, bad);
    }
    mx = __reduce_max_sync(0xffffffffu, mx);
    bad = __reduce_or_sync(0xffffffffu, bad);
    __shared__ uint32_t smx[8], sbad[8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        smx[warp] = mx;
        sbad[warp] = bad;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t m = 0, b = 0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
            m = max(m, smx[w]);
            b |= sbad[w];
        }
        atomicMax(&ws->absmax_bits, m);
        if (b) atomicOr(&ws->nonfinite, 1u);
    }
}

// Magnitude index of one weight: the number of boundaries not above |w|.
// Boundaries are positive fp32 values, so they compare like their bit
// patterns; |w| is compared as bits too (a NaN counts as large and is
// reported separately).  q_max = 7 uses a three-step binary search, q_max = 3
// a two-step one.
template <int QMAX>
__device__ __forceinline__ uint32_t magnitude(uint32_t u, const uint32_t (&t)[8])
{
    if constexpr (QMAX == 7) {
        const bool b2 = u >= t[3];
        const uint32_t t1 = b2 ? t[5] : t[1];
        const bool b1 = u >= t1;
        const uint32_t t0 = b2 ? (b1 ? t[6] : t[4]) : (b1 ? t[2] : t[0]);
        return (b2 ? 4u : 0u) + (b1 ? 2u : 0u) + (u >= t0 ? 1u : 0u);
    } else {
        const bool b1 = u >= t[1];
        const uint32_t t0 = b1 ? t[2] : t[0];
        return (b1 ? 2u : 0u) + (u >= t0 ? 1u : 0u);
    }
}

template <int BITS>
__device__ __forceinline__ uint32_t code_of(uint32_t bits, uint32_t m)
{
    // sign bit only for negative weights that did not round to zero
    const uint32_t sign = (bits >> (32 - BITS)) & (1u << (BITS - 1));
    return m != 0 ? (m | sign) : 0u;
}

// 4-bit: each thread turns 8 consecutive weights into one 32-bit word
// (k even in the low nibble of each byte).
__global__ void __launch_bounds__(256) quantize4_kernel(const float4* __restrict__ W, int64_t nwords,
                                                        QuantParams p, uint32_t* __restrict__ out,
                                                        Workspace* ws)
{
    uint32_t t[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) t[j] = __float_as_uint(p.thresh[j]);
    uint32_t umax = 0;                       // largest |w| bit pattern seen (non-finite check)
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nwords; i += stride) {
        const float4 a = ld_stream(W + 2 * i);
        const float4 b = ld_stream(W + 2 * i + 1);
        const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        uint32_t word = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t bits = __float_as_uint(v[e]);
            const uint32_t u = bits & 0x7fffffffu;
            umax = max(umax, u);
            word += code_of<4>(bits, magnitude<7>(u, t)) << (4 * e);   // disjoint nibbles: add = or
        }
        out[i] = word;
    }
    if (p.check_nonfinite) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0x7f800000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

// 3-bit: each thread packs one group of 32 weights into 12 bytes.
__global__ void __launch_bounds__(256) quantize3_kernel(const float4* __restrict__ W, int64_t ngroups,
                                                        QuantParams p, uint32_t* __restrict__ out,
                                                        Workspace* ws)
{
    uint32_t t[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) t[j] = __float_as_uint(p.thresh[j]);
    uint32_t umax = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < ngroups; g += stride) {
        uint32_t w0 = 0, w1 = 0, w2 = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {            // 4 weights = pairs 2q, 2q+1
            const float4 a = ld_stream(W + 8 * g + q);
            const float v[4] = {a.x, a.y, a.z, a.w};
            uint32_t c[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t bits = __float_as_uint(v[e]);
                const uint32_t u = bits & 0x7fffffffu;
                umax = max(umax, u);
                c[e] = code_of<3>(bits, magnitude<3>(u, t));
            }
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int pair = 2 * q + h;
                const uint32_t f = c[2 * h] | (c[2 * h + 1] << 3);
                if (pair < 15) {
                    const uint32_t sh = f << (6 * (pair % 5));
                    if (pair / 5 == 0) w0 |= sh;
                    else if (pair / 5 == 1) w1 |= sh;
                    else w2 |= sh;
                } else {
                    w0 |= (f & 3u) << 30;
                    w1 |= ((f >> 2) & 3u) << 30;
                    w2 |= ((f >> 4) & 3u) << 30;
                }
            }
        }
        out[3 * g + 0] = w0;
        out[3 * g + 1] = w1;
        out[3 * g + 2] = w2;
    }
    if (p.check_nonfinite) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0x7f800000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

// 8-bit: each thread turns 16 consecutive weights into 16 code bytes.  The
// 127 boundaries live in shared memory (as bit patterns, with +Inf appended)
// and a seven-step binary search counts those not above |w|.
__global__ void __launch_bounds__(256) quantize8_kernel(const float4* __restrict__ W, int64_t n16,
                                                        QuantParams p, uint4* __restrict__ out,
                                                        Workspace* ws)
{
    __shared__ uint32_t t[128];
    if (threadIdx.x < 128) t[threadIdx.x] = threadIdx.x < 127 ? __float_as_uint(p.thresh[threadIdx.x]) : 0x7f800000u;
    __syncthreads();
    uint32_t umax = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += stride) {
        float4 v4[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) v4[j] = ld_stream(W + 4 * i + j);
        uint32_t word[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const float v[4] = {v4[j].x, v4[j].y, v4[j].z, v4[j].w};
            uint32_t wd = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t bits = __float_as_uint(v[e]);
                const uint32_t u = bits & 0x7fffffffu;
                umax = max(umax, u);
                uint32_t m = 0;
#pragma unroll
                for (int step = 64; step >= 1; step >>= 1)
                    if (u >= t[m + step - 1]) m += step;
                wd |= code_of<8>(bits, m) << (8 * e);
            }
            word[j] = wd;
        }
        out[i] = make_uint4(word[0], word[1], word[2], word[3]);
    }
    if (p.check_nonfinite) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0x7f800000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

int grid_for(int64_t items, int threads)
{
    const int sms = sm_count() > 0 ? sm_count() : 148;
    const int64_t need = (items + threads - 1) / threads;
    const int64_t cap = (int64_t)sms * 8;
    return (int)(need < cap ? (need > 0 ? need : 1) : cap);
}

}  // namespace

cudaError_t launch_absmax(const float* W, int64_t count, Workspace* ws, cudaStream_t s)
{
    const int64_t n4 = count / 4;   // count is a multiple of 128
    absmax_kernel<<<grid_for(n4 / 4, 256), 256, 0, s>>>(reinterpret_cast<const float4*>(W), n4, ws);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const float* W, int64_t N, int64_t K, const QuantParams& p,
                            uint8_t* codes, Workspace* ws, cudaStream_t s)
{
    const int64_t total = N * K;
    if (p.bits == 8) {
        const int64_t n16 = total / 16;
        quantize8_kernel<<<grid_for(n16, 256), 256, 0, s>>>(
            reinterpret_cast<const float4*>(W), n16, p, reinterpret_cast<uint4*>(codes), ws);
    } else if (p.bits == 4) {
        const int64_t nwords = total / 8;
        quantize4_kernel<<<grid_for(nwords, 256), 256, 0, s>>>(
            reinterpret_cast<const float4*>(W), nwords, p, reinterpret_cast<uint32_t*>(codes), ws);
    } else {
        const int64_t ngroups = total / 32;
        quantize3_kernel<<<grid_for(ngroups, 256), 256, 0, s>>>(
            reinterpret_cast<const float4*>(W), ngroups, p, reinterpret_cast<uint32_t*>(codes), ws);
    }
    return cudaGetLastError();
}

}  // namespace logq
