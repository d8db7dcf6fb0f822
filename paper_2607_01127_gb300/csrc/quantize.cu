// absmax reduction and quantise + pack kernels (paper Eq. (1), Sec. 3.2 w_max).
//
// Both kernels stream fp32 W once with 16-byte loads that bypass L1.
// The quantiser assigns m = #{ j : |w| >= thresh[j] } against the fp32
// decision boundaries of the codebook (rounded up from fp64), which for fp32
// weights equals round(log_b|w| + s) clamped to [0, q_max].
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "internal.h"

namespace logq {
namespace {

struct QuantEst {
    uint32_t t2[8];     // 2 x the boundaries' bit patterns; 0xffffffff after the last
    uint64_t C;         // fixed-point offset of the level estimate (two's complement)
    uint32_t K;         // fixed-point slope
    uint32_t _pad;
};

struct QuantEst8 {
    uint32_t t2[128];   // 2 x the 127 boundaries' bit patterns; 0xffffffff at 127
    uint32_t corr[64];  // log2(1 + f) - f (lower bound over each 1/64 of f), in units of 2^-24
    uint64_t C;         // fixed-point offset (two's complement), units of 2^-40 of a level
    uint32_t K;         // fixed-point slope
    uint32_t _pad;
};

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

// 4-bit with the level estimated from the weight's bit pattern.  The bit
// pattern u of a positive normal float, read as an integer, is a piecewise-linear
// log2: u / 2^23 - 127 = e + f, below log2 by at most 0.0861.  With the
// boundaries geometric (ratio b = 2^lambda, lambda >= 0.12), the fixed-point
// value floor(((2u - U0) K + C) / 2^32), a little below the level count the
// real log2 would give, is the true count m or m - 1; one comparison with the
// boundary m_est decides: m = m_est + (|w| >= thresh[m_est]).  The decision is
// the boundary comparison itself, so the codes equal quantize4_kernel's.  The
// host sets K, C and the guards (first boundary normal, lambda in [0.12, 3]).
template <bool CHECK>
__global__ void __launch_bounds__(256) quantize4e_kernel(const float4* __restrict__ W, int64_t nwords,
                                                         const __grid_constant__ QuantEst q,
                                                         uint32_t* __restrict__ out, Workspace* ws)
{
    __shared__ uint32_t t2[8];
    if (threadIdx.x < 8) t2[threadIdx.x] = q.t2[threadIdx.x];
    __syncthreads();
    uint32_t umax = 0;                       // largest 2|w| bit pattern seen (non-finite check)
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nwords; i += stride) {
        const float4 a = ld_stream(W + 2 * i);
        const float4 b = ld_stream(W + 2 * i + 1);
        const float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        uint32_t mword = 0, sword = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const uint32_t bits = __float_as_uint(v[e]);
            const uint32_t u2 = bits << 1;   // 2|w|: the sign bit drops out
            if (CHECK) umax = max(umax, u2);
            const uint64_t p = (uint64_t)u2 * q.K + q.C;
            const int mh = __vimin_s32_relu((int)(uint32_t)(p >> 32), 7);
            mword |= ((uint32_t)mh + (u2 >= t2[mh] ? 1u : 0u)) << (4 * e);
            sword |= (bits >> 31) << (4 * e + 3);
        }
        // a sign bit only on nibbles whose magnitude is not 0 (m + 7 carries into bit 3)
        out[i] = mword | (sword & (mword + 0x77777777u) & 0x88888888u);
    }
    if (CHECK) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0xff000000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

// 8-bit with the level estimated as in quantize4e_kernel, the linear log2 of
// the bit pattern corrected by a 64-entry table over the top 6 mantissa bits
// (a lower bound of log2(1 + f) - f on each interval, so the estimate stays
// below log2 by at most 0.0069) and a 40-bit fixed point (127 levels): for
// boundary ratios 2^lambda with lambda >= 0.01 the estimate is the true count
// m or m - 1 and one comparison with the fp32 boundary decides.
template <bool CHECK>
__global__ void __launch_bounds__(256) quantize8e_kernel(const float4* __restrict__ W, int64_t n16,
                                                         const __grid_constant__ QuantEst8 q,
                                                         uint4* __restrict__ out, Workspace* ws)
{
    __shared__ uint32_t t2[128];
    __shared__ uint32_t corr[64];
    if (threadIdx.x < 128) t2[threadIdx.x] = q.t2[threadIdx.x];
    if (threadIdx.x < 64) corr[threadIdx.x] = q.corr[threadIdx.x];
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
            uint32_t mword = 0, sword = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t bits = __float_as_uint(v[e]);
                const uint32_t u2 = bits << 1;
                if (CHECK) umax = max(umax, u2);
                const uint64_t p = (uint64_t)(u2 + corr[(u2 >> 18) & 63]) * q.K + q.C;
                const int mh = __vimin_s32_relu((int)(uint32_t)(p >> 32) >> 8, 127);
                mword |= ((uint32_t)mh + (u2 >= t2[mh] ? 1u : 0u)) << (8 * e);
                sword |= (bits >> 31) << (8 * e + 7);
            }
            word[j] = mword | (sword & (mword + 0x7f7f7f7fu) & 0x80808080u);
        }
        out[i] = make_uint4(word[0], word[1], word[2], word[3]);
    }
    if (CHECK) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0xff000000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

// 3-bit: each thread packs one group of 32 weights into three words (the
// layout in logq.h).  A warp first copies its 32 consecutive groups (4 KiB) from
// global memory with coalesced 16-byte loads (consecutive lanes on consecutive
// 16 bytes) into its own shared-memory stage, and each lane then reads back its
// group's eight 16-byte pieces; the stage is swizzled (piece q of group g at
// g * 8 + (q ^ (g & 7))) so that both the stores and the reads are free of bank
// conflicts.
__global__ void __launch_bounds__(256) quantize3_kernel(const float4* __restrict__ W, int64_t ngroups,
                                                        QuantParams p, uint32_t* __restrict__ out,
                                                        Workspace* ws)
{
    __shared__ float4 stage[8][256];
    uint32_t t[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) t[j] = __float_as_uint(p.thresh[j]);
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    float4* st = stage[wid];
    uint32_t umax = 0;
    const int64_t wstride = (int64_t)gridDim.x * 8 * 32;          // groups per sweep of all warps
    for (int64_t gb = ((int64_t)blockIdx.x * 8 + wid) * 32; gb < ngroups; gb += wstride) {
        const int64_t left = ngroups - gb;
        const int nf = (int)((left < 32 ? left : 32) * 8);         // 16-byte pieces of this batch
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int f = i * 32 + lane;
            const int gl = f >> 3, q = f & 7;
            st[gl * 8 + (q ^ (gl & 7))] = (f < nf) ? ld_stream(W + gb * 8 + f) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        __syncwarp();
        if (lane < nf / 8) {
            uint32_t w0 = 0, w1 = 0, w2 = 0;
#pragma unroll
            for (int q = 0; q < 8; ++q) {            // 4 weights = pairs 2q, 2q+1
                const float4 a = st[lane * 8 + (q ^ (lane & 7))];
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
            const int64_t g = gb + lane;
            out[3 * g + 0] = w0;
            out[3 * g + 1] = w1;
            out[3 * g + 2] = w2;
        }
        __syncwarp();                               // the stage is refilled next sweep
    }
    if (p.check_nonfinite) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0x7f800000u ? 1u : 0u);
        if (bad && (threadIdx.x & 31) == 0) atomicOr(&ws->nonfinite, 1u);
    }
}

// 3-bit with the level estimated as in quantize4e_kernel (q_max = 3; the same
// fixed point and guards).  Each warp streams batches of 32 consecutive groups
// (4 KiB) into two alternating shared-memory stages with asynchronous 16-byte
// copies (swizzled as in quantize3_kernel), so the next batch is in flight while
// the lanes code the current one.  Each weight adds m + 4 * sign into its 3-bit
// slot of the group's word (weights 0-29: word e / 10, slot e % 10, which is the
// layout's field of pair e / 2); the sign is then cleared in every slot whose
// magnitude is 0 at once: (m + 3) carries into the slot's bit 2 exactly when
// m != 0, and never out of the slot.  Weights 30 and 31 (pair 15, split over
// the three words' top bits) are coded one by one.  The codes equal
// quantize3_kernel's bit for bit.
constexpr int kQ3eThreads = 128;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

template <bool CHECK>
__global__ void __launch_bounds__(kQ3eThreads) quantize3e_kernel(const float4* __restrict__ W, int64_t ngroups,
                                                                 const __grid_constant__ QuantEst q,
                                                                 uint32_t* __restrict__ out, Workspace* ws)
{
    constexpr int kWarps = kQ3eThreads / 32;
    __shared__ float4 stage[kWarps][2][256];
    __shared__ uint32_t t2[4];
    if (threadIdx.x < 4) t2[threadIdx.x] = q.t2[threadIdx.x];
    __syncthreads();
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t umax = 0;                                             // largest 2|w| bit pattern seen
    constexpr uint32_t kLow = 0x1B6DB6DBu;                        // 0b011 in each of 10 slots
    constexpr uint32_t kBit2 = 0x24924924u;                       // 0b100 in each of 10 slots
    const int64_t wstride = (int64_t)gridDim.x * kWarps * 32;     // groups per sweep of all warps
    // copies of the batch at gb into stage b (pieces past the end are not copied:
    // only lanes whose group exists read the stage)
    auto issue = [&](int b, int64_t gb) {
        const int64_t left = ngroups - gb;
        const int nf = (int)((left < 32 ? left : 32) * 8);
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(&stage[wid][b][0]);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int f = i * 32 + lane;
            const int gl = f >> 3, qq = f & 7;
            if (f < nf) cp_async16(base + 16u * (uint32_t)(gl * 8 + (qq ^ (gl & 7))), W + gb * 8 + f);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    int64_t gb = ((int64_t)blockIdx.x * kWarps + wid) * 32;
    if (gb < ngroups) issue(0, gb);
    for (int b = 0; gb < ngroups; b ^= 1) {
        const int64_t gn = gb + wstride;
        if (gn < ngroups) issue(b ^ 1, gn);
        else asm volatile("cp.async.commit_group;" ::: "memory");   // keeps one group per batch
        asm volatile("cp.async.wait_group 1;" ::: "memory");         // this batch has landed
        __syncwarp();
        const float4* st = stage[wid][b];
        const int64_t left = ngroups - gb;
        if (lane < (left < 32 ? left : 32)) {
            uint32_t v[3] = {0u, 0u, 0u};
            uint32_t c30 = 0, c31 = 0;
#pragma unroll
            for (int qq = 0; qq < 8; ++qq) {
                const float4 a = st[lane * 8 + (qq ^ (lane & 7))];
                const float w4[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = 4 * qq + i;
                    const uint32_t bits = __float_as_uint(w4[i]);
                    const uint32_t u2 = bits << 1;                  // 2|w|: the sign bit drops out
                    if (CHECK) umax = max(umax, u2);
                    const uint64_t pe = (uint64_t)u2 * q.K + q.C;
                    const int mh = __vimin_s32_relu((int)(uint32_t)(pe >> 32), 3);
                    const uint32_t val = (uint32_t)mh + (u2 >= t2[mh] ? 1u : 0u) + ((bits >> 31) << 2);
                    if (e < 30) v[e / 10] += val << (3 * (e % 10));  // disjoint slots: add = or
                    else if (e == 30) c30 = val;
                    else c31 = val;
                }
            }
#pragma unroll
            for (int j = 0; j < 3; ++j) {
                const uint32_t lo = v[j] & kLow;
                v[j] = lo | (v[j] & ((lo + kLow) & kBit2));
            }
            c30 = (c30 & 3u) | (c30 & (((c30 & 3u) + 3u) & 4u));
            c31 = (c31 & 3u) | (c31 & (((c31 & 3u) + 3u) & 4u));
            const uint32_t f15 = c30 | (c31 << 3);
            const int64_t g = gb + lane;
            out[3 * g + 0] = v[0] | ((f15 & 3u) << 30);
            out[3 * g + 1] = v[1] | (((f15 >> 2) & 3u) << 30);
            out[3 * g + 2] = v[2] | (((f15 >> 4) & 3u) << 30);
        }
        __syncwarp();                                  // stage b is refilled two batches on
        gb = gn;
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (CHECK) {
        const uint32_t bad = __reduce_or_sync(0xffffffffu, umax >= 0xff000000u ? 1u : 0u);
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

// Fixed-point slope and offset of the level estimate of quantize4e_kernel and
// quantize3e_kernel, from the 4-bit (q_max = 7) or 3-bit (q_max = 3)
// boundaries; false when the guards fail (the boundary search is used).
//   lambda = log2 of the boundary ratio, from the first and last boundary;
//   estimate(u2) = floor((u2 K + C) / 2^32) with K = round(2^8 / lambda) and
//   C = round(-(log2 t_0 + 127) 2^24 K + (1 - 0.05) 2^32), i.e. the level count
//   from the linear log2 of the bit pattern, biased down by 0.05 of a level so
//   that the rounding of K, C and of the boundaries never lifts it above the
//   true count; the linear log2 lies below log2 by at most 0.0861, i.e.
//   0.0861 / lambda <= 0.72 levels for lambda >= 0.12.
bool estimate_params(const QuantParams& p, QuantEst& q)
{
    if (!((p.bits == 4 && p.qmax == 7) || (p.bits == 3 && p.qmax == 3))) return false;
    const int last = p.qmax - 1;
    const double t0 = p.thresh[0], tl = p.thresh[last];
    if (!(t0 >= 1.1754943508222875e-38) || !(tl > t0) || !isfinite(tl)) return false;
    const double l0 = log2(t0);
    const double lambda = (log2(tl) - l0) / (double)last;
    if (!(lambda >= 0.12) || !(lambda <= 3.0)) return false;
    const double k = nearbyint(256.0 / lambda);
    q.K = (uint32_t)k;
    q.C = (uint64_t)(int64_t)nearbyint(-(l0 + 127.0) * 16777216.0 * k + 0.95 * 4294967296.0);
    for (int j = 0; j < 8; ++j) {
        uint32_t b = 0;
        if (j < p.qmax) memcpy(&b, &p.thresh[j], 4);
        q.t2[j] = j < p.qmax ? 2u * b : 0xffffffffu;
    }
    q._pad = 0;
    return true;
}

// quantize8e_kernel's parameters (lambda and the table as above, K = round(2^16 /
// lambda), C = round(-(log2 t_0 + 127) 2^24 K + 0.95 2^40)); false when the guards
// fail: first boundary below 2^-120 (subnormal weights plus the table's
// correction must stay below it) or lambda outside [0.01, 4].
bool estimate_params8(const QuantParams& p, QuantEst8& q)
{
    if (p.bits != 8 || p.qmax != 127) return false;
    const double t0 = p.thresh[0], tl = p.thresh[126];
    if (!(t0 >= 7.52316384526264e-37) || !(tl > t0) || !isfinite(tl)) return false;   // 2^-120
    const double l0 = log2(t0);
    const double lambda = (log2(tl) - l0) / 126.0;
    if (!(lambda >= 0.01) || !(lambda <= 4.0)) return false;
    const double k = nearbyint(65536.0 / lambda);
    q.K = (uint32_t)k;
    q.C = (uint64_t)(int64_t)nearbyint(-(l0 + 127.0) * 16777216.0 * k + 0.95 * 1099511627776.0);
    for (int j = 0; j < 127; ++j) {
        uint32_t b;
        memcpy(&b, &p.thresh[j], 4);
        q.t2[j] = 2u * b;
    }
    q.t2[127] = 0xffffffffu;
    for (int i = 0; i < 64; ++i) {
        const double f0 = i / 64.0, f1 = (i + 1) / 64.0;
        const double g0 = log2(1.0 + f0) - f0, g1 = log2(1.0 + f1) - f1;   // concave: minimum at an end
        q.corr[i] = (uint32_t)floor(16777216.0 * (g0 < g1 ? g0 : g1));
    }
    q._pad = 0;
    return true;
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
        QuantEst8 q;
        if (estimate_params8(p, q)) {
            if (p.check_nonfinite)
                quantize8e_kernel<true><<<grid_for(n16, 256), 256, 0, s>>>(
                    reinterpret_cast<const float4*>(W), n16, q, reinterpret_cast<uint4*>(codes), ws);
            else
                quantize8e_kernel<false><<<grid_for(n16, 256), 256, 0, s>>>(
                    reinterpret_cast<const float4*>(W), n16, q, reinterpret_cast<uint4*>(codes), ws);
        } else {
            quantize8_kernel<<<grid_for(n16, 256), 256, 0, s>>>(
                reinterpret_cast<const float4*>(W), n16, p, reinterpret_cast<uint4*>(codes), ws);
        }
    } else if (p.bits == 4) {
        const int64_t nwords = total / 8;
        QuantEst q;
        if (estimate_params(p, q)) {
            if (p.check_nonfinite)
                quantize4e_kernel<true><<<grid_for(nwords, 256), 256, 0, s>>>(
                    reinterpret_cast<const float4*>(W), nwords, q, reinterpret_cast<uint32_t*>(codes), ws);
            else
                quantize4e_kernel<false><<<grid_for(nwords, 256), 256, 0, s>>>(
                    reinterpret_cast<const float4*>(W), nwords, q, reinterpret_cast<uint32_t*>(codes), ws);
        } else {
            quantize4_kernel<<<grid_for(nwords, 256), 256, 0, s>>>(
                reinterpret_cast<const float4*>(W), nwords, p, reinterpret_cast<uint32_t*>(codes), ws);
        }
    } else {
        const int64_t ngroups = total / 32;
        // 32 KiB of staging per CTA: at most six resident per SM
        const int sms = sm_count() > 0 ? sm_count() : 148;
        int grid3 = grid_for(ngroups, 256);
        if (grid3 > sms * 6) grid3 = sms * 6;
        QuantEst q;
        if (estimate_params(p, q)) {
            // 32 KiB of stages per 128-thread CTA: six resident per SM
            int grid3e = (int)((ngroups + kQ3eThreads - 1) / kQ3eThreads);
            if (grid3e > sms * 6) grid3e = sms * 6;
            if (p.check_nonfinite)
                quantize3e_kernel<true><<<grid3e, kQ3eThreads, 0, s>>>(
                    reinterpret_cast<const float4*>(W), ngroups, q, reinterpret_cast<uint32_t*>(codes), ws);
            else
                quantize3e_kernel<false><<<grid3e, kQ3eThreads, 0, s>>>(
                    reinterpret_cast<const float4*>(W), ngroups, q, reinterpret_cast<uint32_t*>(codes), ws);
        } else {
            quantize3_kernel<<<grid3, 256, 0, s>>>(
                reinterpret_cast<const float4*>(W), ngroups, p, reinterpret_cast<uint32_t*>(codes), ws);
        }
    }
    return cudaGetLastError();
}

}  // namespace logq
