// Energy-based effective range (paper Sec. 3.2, Eq. (5)): the smallest data
// value t with  sum_{|w_i| <= t} w_i^2  >=  eps * sum_i w_i^2,  and w_max = max |w_i|.
//
// w_min is an order statistic, so it is found by a radix selection over the
// 31-bit pattern u = bits(|w|) (non-negative floats order like their bit
// patterns), three streaming passes over W:
//   level 1: bucket u >> 23 (the exponent), 256 buckets;
//   level 2: within the level-1 exponent, (u >> 11) & 0xfff, 4096 buckets;
//   level 3: within the level-2 prefix u >> 11, u & 0x7ff, one value each.
// Every value of a bucket shares its exponent e, so w^2 = m^2 * 2^(2e - 46)
// with m the 24-bit significand: a bucket's energy is kept exactly as two
// 64-bit integer sums (the high and low 24 bits of m^2), accumulated with
// integer atomics in shared memory and flushed with integer atomics to global
// memory, so the per-bucket sums do not depend on the order of the additions.
// At level 1, where every weight lands in one of a few hot buckets, each warp
// keeps its own copy of the 256 buckets and takes the distinct exponents of
// its 32 values one at a time: their lanes add their parts with a warp
// reduction (exact: 32 parts of 24 bits fit in 32 bits) and one lane adds the
// sums to the warp's copy, without atomics; the copies are summed in a fixed
// order at the end of the pass.
// When eps is not tiny (eps > n * 2^-59, always so for the paper's 4e-3 and
// 1e-6) level 1 instead follows an absmax pass and counts only the 31
// exponents at and below that of w_max: each lane adds its values' m^2 to its
// own 64-bit cells in shared memory (no collectives, no atomics, no fp64) and
// folds them into registers every 256 values, long before a cell or a fold can
// overflow.  Values below the window go to bucket 0 in the unit of bucket 1
// (m^2 shifted right by twice the exponent difference; the truncation is below
// 2^-106 of the total energy per value).  Each of them holds less than 2^-60
// of the total energy, so their share is below n * 2^-60 < eps and the
// crossing lies inside the window.
// After each pass one CTA converts the bucket sums to fp64 and scans them in
// ascending order from the energy below the bucket's prefix (a fixed-order
// parallel scan): the first bucket whose cumulative share cum / total reaches
// eps is the next prefix.  Level 1 also takes w_max and the non-finite flag.
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace logq {
namespace {

constexpr int kHistThreads = 256;
constexpr int kScanThreads = 256;
constexpr int kUnroll = 4;                       // float4 loads in flight per thread

template <int LEVEL> struct Level;
template <> struct Level<1> { static constexpr int NB = 256, COPIES = kHistThreads / 32; };
template <> struct Level<2> { static constexpr int NB = 4096, COPIES = 1; };
template <> struct Level<3> { static constexpr int NB = 2048, COPIES = 1; };
static_assert(sizeof(EnergyState::hi) / sizeof(EnergyState::hi[0]) >= 4096, "bucket arrays");

__device__ __forceinline__ float4 ld_stream4(const float4* p)
{
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}

// m^2 of a finite |w| pattern, split into its high and low 24 bits.
__device__ __forceinline__ void msq_parts(uint32_t u, uint32_t& hi, uint32_t& lo)
{
    const uint32_t mant = u & 0x7fffffu;
    const uint32_t m = (u >> 23) ? (mant | 0x800000u) : mant;      // subnormals: no implicit bit
    const unsigned long long sq = (unsigned long long)m * m;         // < 2^48
    hi = (uint32_t)(sq >> 24);
    lo = (uint32_t)(sq & 0xffffffull);
}

template <int LEVEL>
__device__ __forceinline__ void add_one(uint32_t u, uint32_t prefix, unsigned long long* hi,
                                        unsigned long long* lo)
{
    const bool finite = u < 0x7f800000u;
    if constexpr (LEVEL == 1) {
        // every lane of the warp takes part (the loop trip count is uniform)
        uint32_t h = 0, l = 0;
        if (finite) msq_parts(u, h, l);
        const uint32_t b = u >> 23;
        // one round per distinct exponent in the warp (a handful for weights):
        // the lanes of that exponent add their parts, the first of them adds
        // the sums to this warp's copy of the buckets
        const uint32_t lane = threadIdx.x & 31;
        uint32_t todo = 0xffffffffu;
        while (todo) {
            const int first = __ffs(todo) - 1;
            const uint32_t bb = __shfl_sync(0xffffffffu, b, first);
            const uint32_t peers = __ballot_sync(0xffffffffu, b == bb);
            const uint32_t sh = __reduce_add_sync(0xffffffffu, b == bb ? h : 0u);
            const uint32_t sl = __reduce_add_sync(0xffffffffu, b == bb ? l : 0u);
            if (lane == (uint32_t)first && (sh | sl)) {
                hi[bb] += sh;
                lo[bb] += sl;
            }
            todo &= ~peers;
        }
        __syncwarp();
    } else {
        const bool in = finite && (LEVEL == 2 ? (u >> 23) == prefix : (u >> 11) == prefix);
        if (!in) return;
        const uint32_t b = LEVEL == 2 ? ((u >> 11) & 0xfffu) : (u & 0x7ffu);
        uint32_t h, l;
        msq_parts(u, h, l);
        if (h | l) {
            atomicAdd(&hi[b], (unsigned long long)h);
            atomicAdd(&lo[b], (unsigned long long)l);
        }
    }
}

template <int LEVEL>
__global__ void __launch_bounds__(kHistThreads) energy_hist_kernel(const float4* __restrict__ W, int64_t n4,
                                                                   EnergyState* st, Workspace* ws)
{
    constexpr int NB = Level<LEVEL>::NB, COPIES = Level<LEVEL>::COPIES;
    extern __shared__ unsigned long long hist[];              // [COPIES][2][NB]
    for (int i = threadIdx.x; i < 2 * NB * COPIES; i += kHistThreads) hist[i] = 0;
    __syncthreads();
    unsigned long long* hi = hist + (COPIES > 1 ? (threadIdx.x >> 5) * 2 * NB : 0);
    unsigned long long* lo = hi + NB;
    const uint32_t prefix = LEVEL == 1 ? 0u : st->prefix;
    uint32_t umax = 0, bad = 0;
    auto take = [&](const float4& v) {
        const uint32_t u[4] = {__float_as_uint(v.x) & 0x7fffffffu, __float_as_uint(v.y) & 0x7fffffffu,
                               __float_as_uint(v.z) & 0x7fffffffu, __float_as_uint(v.w) & 0x7fffffffu};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            if (LEVEL == 1) {
                const bool nf = u[e] >= 0x7f800000u;
                bad |= nf ? 1u : 0u;
                umax = max(umax, nf ? 0u : u[e]);
            }
            add_one<LEVEL>(u[e], prefix, hi, lo);
        }
    };
    // Whole rounds of kUnroll loads are taken by every thread of the grid
    // (uniform trip count, so whole warps stay converged); the rest follows.
    const int64_t nthreads = (int64_t)gridDim.x * kHistThreads;
    const int64_t gtid = (int64_t)blockIdx.x * kHistThreads + threadIdx.x;
    const int64_t rounds = n4 / (nthreads * kUnroll);
    for (int64_t r = 0; r < rounds; ++r) {
        const int64_t base = r * nthreads * kUnroll + gtid;
        float4 v[kUnroll];
#pragma unroll
        for (int j = 0; j < kUnroll; ++j) v[j] = ld_stream4(W + base + j * nthreads);
#pragma unroll
        for (int j = 0; j < kUnroll; ++j) take(v[j]);
    }
    for (int64_t i0 = rounds * nthreads * kUnroll; i0 < n4; i0 += nthreads) {
        // tail: whole warps iterate while any of their lanes has an element
        const int64_t i = i0 + gtid;
        const float4 v = i < n4 ? ld_stream4(W + i) : make_float4(0.f, 0.f, 0.f, 0.f);
        take(v);
    }
    if (LEVEL == 1) {
        bad = __reduce_or_sync(0xffffffffu, bad);
        umax = __reduce_max_sync(0xffffffffu, umax);
        if ((threadIdx.x & 31) == 0) {
            if (bad) atomicOr(&ws->nonfinite, 1u);
            atomicMax(&ws->absmax_bits, umax);
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < NB; i += kHistThreads) {
        unsigned long long sh = 0, sl = 0;
#pragma unroll
        for (int c = 0; c < COPIES; ++c) {
            sh += hist[c * 2 * NB + i];
            sl += hist[c * 2 * NB + NB + i];
        }
        if (sh) atomicAdd(&st->hi[i], sh);
        if (sl) atomicAdd(&st->lo[i], sl);
    }
}

// 2^k as a double (normal range: k in [-1022, 1023]).
__device__ __forceinline__ double pow2(int k) { return __longlong_as_double((long long)(1023 + k) << 52); }

constexpr int kWin = 32;            // bucket 0: below the window; 1..31: exponent fields e_hi-30 .. e_hi
constexpr int kFlushRounds = 16;    // 16 rounds x 16 values = 256 values per lane between folds

// Level 1 after an absmax pass: exponent window of w_max, lane-private cells.
__global__ void __launch_bounds__(kHistThreads) energy_window_kernel(const float4* __restrict__ W, int64_t n4,
                                                                     EnergyState* st, const Workspace* ws)
{
    extern __shared__ unsigned long long cells[];     // [warp][kWin][32 lanes]: sums of m^2
    __shared__ unsigned long long wsum[kHistThreads / 32][2][kWin];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned long long* ce = cells + warp * kWin * 32;
    for (int b = 0; b < kWin; ++b) ce[b * 32 + lane] = 0;
    const int e_lo = (int)(ws->absmax_bits >> 23) - (kWin - 2);     // exponent field of bucket 1
    unsigned long long acc_hi = 0, acc_lo = 0;        // bucket `lane` of this warp, folded so far
    auto fold = [&]() {
        __syncwarp();
        // lane l collects bucket l from every lane's cells (rotated start); a
        // cell holds < 2^56 (256 values of m^2 < 2^48), the 32 of them < 2^61,
        // which is split into its high and low 24-bit parts
        unsigned long long sum = 0;
#pragma unroll 8
        for (int j = 0; j < 32; ++j) sum += ce[lane * 32 + ((j + lane) & 31)];
        acc_hi += sum >> 24;
        acc_lo += sum & 0xffffffull;
        __syncwarp();
        for (int b = 0; b < kWin; ++b) ce[b * 32 + lane] = 0;
        __syncwarp();
    };
    auto take = [&](const float4& v) {
        const uint32_t u[4] = {__float_as_uint(v.x) & 0x7fffffffu, __float_as_uint(v.y) & 0x7fffffffu,
                               __float_as_uint(v.z) & 0x7fffffffu, __float_as_uint(v.w) & 0x7fffffffu};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            if (u[e] >= 0x7f800000u) continue;           // reported by the absmax pass
            const int field = (int)(u[e] >> 23);
            const int d = field - e_lo + 1;
            const uint32_t mant = u[e] & 0x7fffffu;
            const uint32_t m = field ? (mant | 0x800000u) : mant;
            const int sh = d >= 1 ? 0 : 2 * (e_lo - (field ? field : 1));   // below the window
            const unsigned long long sq = (unsigned long long)m * m;
            ce[(d >= 1 ? d : 0) * 32 + lane] += sh < 64 ? (sq >> sh) : 0ull;
        }
    };
    const int64_t nthreads = (int64_t)gridDim.x * kHistThreads;
    const int64_t gtid = (int64_t)blockIdx.x * kHistThreads + threadIdx.x;
    const int64_t rounds = n4 / (nthreads * kUnroll);
    for (int64_t r = 0; r < rounds; ++r) {
        const int64_t base = r * nthreads * kUnroll + gtid;
        float4 v[kUnroll];
#pragma unroll
        for (int j = 0; j < kUnroll; ++j) v[j] = ld_stream4(W + base + j * nthreads);
#pragma unroll
        for (int j = 0; j < kUnroll; ++j) take(v[j]);
        if ((r % kFlushRounds) == kFlushRounds - 1) fold();
    }
    for (int64_t i0 = rounds * nthreads * kUnroll; i0 < n4; i0 += nthreads) {
        const int64_t i = i0 + gtid;
        if (i < n4) take(ld_stream4(W + i));
    }
    fold();
    // per warp: lane l holds bucket l
    wsum[warp][0][lane] = acc_hi;
    wsum[warp][1][lane] = acc_lo;
    __syncthreads();
    if (threadIdx.x < kWin) {
        unsigned long long sh = 0, sl = 0;
        for (int w = 0; w < kHistThreads / 32; ++w) {
            sh += wsum[w][0][threadIdx.x];
            sl += wsum[w][1][threadIdx.x];
        }
        if (sh) atomicAdd(&st->hi[threadIdx.x], sh);
        if (sl) atomicAdd(&st->lo[threadIdx.x], sl);
    }
}

// Scan of the window pass: bucket 0 is the energy below the window (in bucket
// 1's unit), buckets 1..31 the window's exponents.
__global__ void __launch_bounds__(32) energy_scan_window_kernel(EnergyState* st, const Workspace* ws, double eps)
{
    __shared__ double en[kWin];
    const int t = threadIdx.x;
    const int e_lo = (int)(ws->absmax_bits >> 23) - (kWin - 2);
    {
        const int field = t == 0 ? e_lo : e_lo + t - 1;
        double x = 0.0;
        if (field >= 0) {
            const int e = (field ? field : 1) - 127;
            x = ((double)st->hi[t] * 16777216.0 + (double)st->lo[t]) * pow2(2 * e - 46);
        }
        en[t] = x;
    }
    __syncwarp();
    if (t == 0) {
        double total = 0.0;
        for (int b = 0; b < kWin; ++b) total += en[b];
        st->total = total;
        double cum = 0.0;
        int found = -1;
        double before = 0.0;
        const double near = eps * total * (1.0 - 0x1p-40);   // below this the share is surely < eps
        for (int b = 0; b < kWin && found < 0; ++b) {
            const double prev = cum;
            cum += en[b];
            if (en[b] > 0.0 && cum >= near && cum / total >= eps) {
                found = b;
                before = prev;
            }
        }
        if (found <= 0) {
            st->failed = 1;          // not reachable when eps > n * 2^-59
            found = kWin - 1;
        }
        st->below = before;
        st->prefix = (uint32_t)(e_lo + found - 1);   // the exponent field, as level 1 leaves it
    }
}

// One CTA: bucket energies in fp64, ascending inclusive scan from the energy
// below the prefix, first bucket whose share reaches eps.
template <int LEVEL>
__global__ void __launch_bounds__(kScanThreads) energy_scan_kernel(EnergyState* st, double eps)
{
    constexpr int NB = Level<LEVEL>::NB;
    constexpr int PER = NB / kScanThreads;               // buckets per thread, contiguous
    __shared__ double part[2][kScanThreads];
    __shared__ int found;
    const int t = threadIdx.x;
    const uint32_t prefix = st->prefix;
    // exponent field of the level's values: the bucket itself (level 1) or the prefix
    auto efield_of = [&](int b) -> uint32_t {
        return LEVEL == 1 ? (uint32_t)b : (LEVEL == 2 ? prefix : (prefix >> 12));
    };
    auto energy = [&](int b) -> double {
        const uint32_t ef = efield_of(b);
        const int e = (ef ? (int)ef : 1) - 127;
        return ((double)st->hi[b] * 16777216.0 + (double)st->lo[b]) * pow2(2 * e - 46);
    };
    double en[PER];
    double mine = 0.0;
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        en[j] = energy(t * PER + j);
        mine += en[j];
    }
    // fixed-order inclusive scan of the per-thread sums (Hillis-Steele)
    int cur = 0;
    part[0][t] = mine;
    if (t == 0) found = NB;
    __syncthreads();
    for (int off = 1; off < kScanThreads; off <<= 1) {
        const double x = part[cur][t] + (t >= off ? part[cur][t - off] : 0.0);
        part[cur ^ 1][t] = x;
        cur ^= 1;
        __syncthreads();
    }
    if (LEVEL == 1 && t == 0) {
        st->total = part[cur][kScanThreads - 1];
        st->below = 0.0;
    }
    __syncthreads();
    const double total = st->total;
    const double below0 = st->below;
    double cum = below0 + (t > 0 ? part[cur][t - 1] : 0.0);
    double cum_before = 0.0;                             // energy below this thread's crossing bucket
    int mine_found = NB;
    const double near = eps * total * (1.0 - 0x1p-40);   // below this the share is surely < eps
#pragma unroll
    for (int j = 0; j < PER; ++j) {
        const double prev = cum;
        cum += en[j];
        if (mine_found == NB && en[j] > 0.0 && cum >= near && cum / total >= eps) {
            mine_found = t * PER + j;
            cum_before = prev;
        }
    }
    atomicMin(&found, mine_found);
    __syncthreads();
    const int b = found;
    auto publish = [&](int bucket, double below) {
        st->below = below;
        const uint32_t np = LEVEL == 1 ? (uint32_t)bucket
                                       : (LEVEL == 2 ? (prefix << 12) | (uint32_t)bucket : (prefix << 11) | (uint32_t)bucket);
        st->prefix = np;
        if (LEVEL == 3) st->wmin_bits = np;
    };
    if (b < NB) {
        if (t == b / PER) publish(b, cum_before);
    } else if (t == 0) {
        // the share stayed a rounding step short of eps inside the parent
        // bucket: the parent's last non-empty value closes it
        int last = 0;
        double run = below0, before = below0;
        for (int i = 0; i < NB; ++i) {
            const double x = energy(i);
            if (x > 0.0) {
                last = i;
                before = run;
            }
            run += x;
        }
        publish(last, before);
    }
}

template <int LEVEL>
cudaError_t hist(const float* W, int64_t n4, EnergyState* st, Workspace* ws, int grid, cudaStream_t s)
{
    constexpr size_t smem = 2 * sizeof(unsigned long long) * Level<LEVEL>::NB * Level<LEVEL>::COPIES;
    static int configured[64] = {0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev] && smem > 48 * 1024) {
        e = cudaFuncSetAttribute(energy_hist_kernel<LEVEL>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    configured[dev] = 1;
    energy_hist_kernel<LEVEL><<<grid, kHistThreads, smem, s>>>(reinterpret_cast<const float4*>(W), n4, st, ws);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_energy_range(const float* W, int64_t count, double eps, EnergyState* st, Workspace* ws,
                                cudaStream_t s)
{
    const int64_t n4 = count / 4;
    const int sms = sm_count() > 0 ? sm_count() : 148;
    int64_t want = (n4 + kHistThreads * kUnroll - 1) / (kHistThreads * kUnroll);
    const int64_t cap = 3 * (int64_t)sms;
    const int grid = (int)(want < cap ? (want > 0 ? want : 1) : cap);
    cudaError_t e;
    const size_t bucket_bytes = sizeof st->hi + sizeof st->lo;
    if ((e = cudaMemsetAsync(st, 0, sizeof(EnergyState), s)) != cudaSuccess) return e;
    if (eps > (double)count * ldexp(1.0, -59)) {
        // the crossing lies within 31 exponents of w_max's
        if ((e = launch_absmax(W, count, ws, s)) != cudaSuccess) return e;
        constexpr size_t smem = (size_t)(kHistThreads / 32) * kWin * 32 * sizeof(unsigned long long);
        static int configured[64] = {0};
        int dev = 0;
        if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
        if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
        if (!configured[dev]) {
            e = cudaFuncSetAttribute(energy_window_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            configured[dev] = 1;
        }
        energy_window_kernel<<<grid, kHistThreads, smem, s>>>(reinterpret_cast<const float4*>(W), n4, st, ws);
        energy_scan_window_kernel<<<1, 32, 0, s>>>(st, ws, eps);
    } else {
        if ((e = hist<1>(W, n4, st, ws, grid, s)) != cudaSuccess) return e;
        energy_scan_kernel<1><<<1, kScanThreads, 0, s>>>(st, eps);
    }
    // levels 2 and 3 re-stream W and keep only the selected prefix
    if ((e = cudaMemsetAsync(st->hi, 0, bucket_bytes, s)) != cudaSuccess) return e;
    if ((e = hist<2>(W, n4, st, ws, grid, s)) != cudaSuccess) return e;
    energy_scan_kernel<2><<<1, kScanThreads, 0, s>>>(st, eps);
    if ((e = cudaMemsetAsync(st->hi, 0, bucket_bytes, s)) != cudaSuccess) return e;
    if ((e = hist<3>(W, n4, st, ws, grid, s)) != cudaSuccess) return e;
    energy_scan_kernel<3><<<1, kScanThreads, 0, s>>>(st, eps);
    return cudaGetLastError();
}

}  // namespace logq
