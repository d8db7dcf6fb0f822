// Decode GEMV / skinny GEMM on CUDA cores: Y[b][n] = sum_k X[b][k] * table[code(n, k)]
// (paper Sec. 3.3: dequantisation by lookup table instead of exponentiation).
//
// Design (CTAs of 8 or 16 warps, see the launch shapes below):
//  * Pair table in shared memory.  Two codes (one byte at 4 bits, one 6-bit
//    field at 3 bits) index a table whose entry is the bf16x2 / f16x2 pair of
//    their dequantised values, signs included.  Each entry occupies a 256-byte
//    row holding one copy per lane, so lane l always reads bank l: the lookups
//    of a warp never conflict.  The table starts the dynamic shared memory at
//    the fixed shared address kTabOff, so the byte offset of an entry,
//    byte << 8 | 4 * lane, is one byte permute (prmt) of the code word and the
//    table base is the load's immediate offset.
//  * Each warp owns a fixed span of K (32 lanes x KW consecutive k) and keeps
//    its activations for that span in registers for the whole kernel; it walks
//    the rows of the CTA's row range, one 16-, 8- or 4-byte coalesced load of
//    codes per lane and row (a warp reads a contiguous 512/256/128-byte run).
//  * fp32 accumulation (mixed-precision fma with bf16/f16 operands), a
//    reduce-scatter across the 32 lanes per round of rows, then a fixed-order
//    sum over the spans in shared memory: results are bit-identical from run
//    to run.
//  * Batch-1 4-bit launches run 8-warp CTAs, two per SM (tiny ones one per
//    SM): with programmatic dependent launch, a CTA of the next launch on the
//    stream starts as soon as one of them leaves, and builds its table and
//    issues its first code loads while the rest of this launch finishes.
//    Other small launches run one 8-warp CTA per SM (room for the next
//    launch's CTAs), other large ones one 16-warp CTA per SM.  Batches of 4
//    and more hold more k per lane where registers allow (one CTA per SM), so
//    that the cross-lane reduction of each row is shared by more multiply-adds.
//  * Where it pays, the CTA's contiguous range of code rows is prefetched into
//    L2 with bulk prefetches at kernel start; an optional warm-up range (the
//    next launch's codes) is prefetched the same way when it is small.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>
#include <string.h>

#include <type_traits>

#include "internal.h"

namespace logq {
namespace {

// Threads per CTA: 256 (two CTAs fit on an SM) for batch-1 4-bit launches,
// small launches and batches of 4 and more, 512 (one per SM, all 16 warps
// sharing one table) for the other large launches.
constexpr int kSmallThreads = 256;
constexpr int kLargeThreads = 512;
constexpr int kTabStride = 256;               // bytes per pair-table entry
// Shared address at which dynamic shared memory starts in a kernel without
// static shared memory: the per-CTA reserved area comes first.
constexpr uint32_t kTabOff = 1024;
constexpr uint32_t kLvlOff = 128;             // levels staged in the free half of table row 0
// Span partials: for batch 1-2 at 4 bits they live in the free upper halves
// of the table's 256 rows (32 KiB), otherwise after the table.
constexpr int kRedBytes = 32 * 1024;
__host__ __device__ constexpr bool red_in_table(int bits, int B) { return bits == 4 && B <= 2; }
constexpr int64_t kPrefetchCap = 1 << 20;     // bytes of codes prefetched per CTA up front
constexpr int kMaxSmem = 256 * kTabStride + kRedBytes;
constexpr int kMaxItems = 4;
// Launches with at least this many bytes of codes run 16 warps per SM (4-bit
// batch 1: as two CTAs): their main loop needs them to keep enough loads in
// flight.  Smaller launches run 8 warps per SM, leaving the other half of the
// SM to the next launch.  Warm-up ranges of this size or more are not
// prefetched.
#ifndef LOGQ_GEMV_SPLIT_BYTES
#define LOGQ_GEMV_SPLIT_BYTES (20 << 20)
#endif
constexpr int64_t kSplitBytes = LOGQ_GEMV_SPLIT_BYTES;
// Batch-1 4-bit launches below this many bytes of codes take 16 k per lane
// (twice the spans, half the activations per lane): their few rows per warp
// finish sooner after the activations arrive.
#ifndef LOGQ_GEMV_TINY_BYTES
#define LOGQ_GEMV_TINY_BYTES (4 << 20)
#endif
constexpr int64_t kTinyBytes = LOGQ_GEMV_TINY_BYTES;
// Tiny batch-1 4-bit launches: CTAs per SM, and whether they prefetch their
// own code rows into L2 (one CTA per SM with the prefetch measured best on the
// 1B decode step; every other batch-1 4-bit launch runs two per SM without it).
#ifndef LOGQ_GEMV_TINY_PER_SM
#define LOGQ_GEMV_TINY_PER_SM 1
#endif
constexpr int kTinyPerSm = LOGQ_GEMV_TINY_PER_SM;
#ifndef LOGQ_GEMV_TINY_OWN_PF
#define LOGQ_GEMV_TINY_OWN_PF 1
#endif
// Shared-memory carveout of the batch-1/2 decode kernels, in percent of the
// maximum: 58 % is 132 KiB, room for two CTAs of 64 KiB (plus their reserved
// 1 KiB).  The rest of the 256 KiB per SM is L1, which also holds the data of
// the code loads in flight, so a larger carveout slows the kernel down; one
// setting for all of them spares the SMs a reconfiguration between launches.
// Batches of 4 and more (two CTAs of up to 97 KiB) take the largest one.
#ifndef LOGQ_GEMV_CARVEOUT
#define LOGQ_GEMV_CARVEOUT 58
#endif

// One matrix of a grouped launch: all items share X, K, B and the code width.
struct GemvItem {
    const uint8_t* codes;
    void* Y;
    int32_t N;
    int32_t cta_begin;    // first CTA of this item
    int32_t cta_count;    // CTAs assigned to it
    int32_t rows_q;       // N / cta_count
    int32_t rows_rem;     // N % cta_count (the first rows_rem CTAs take one more row)
    int32_t _pad;
    uint32_t lvl16[16];   // code-indexed 16-bit levels (low half used)
};

struct GemvParams {
    GemvItem item[kMaxItems];
    int32_t nitems;
    int32_t K;
    int32_t B;
    int32_t y_dtype;
    const uint16_t* X;
    uint32_t* err;        // workspace error word
    int64_t row_bytes;
    int32_t spans;        // S: spans of 32*KW k covering K
    int32_t groups;       // G: warps sharing one span (row-parallel)
    int32_t span_cols;    // warps / G: spans in flight at once
    int32_t chunk_rows;   // rows reduced per shared-memory pass
    const uint8_t* pf;    // optional L2 warm-up range (e.g. the next layer's codes)
    int64_t pf_bytes;
    int64_t pf_share;     // bytes of that range per CTA (multiple of 16)
    int32_t own_pf;       // prefetch the CTA's own code rows into L2 at start
    int32_t _pad;
};

// 8-bit codes: their 256 code-indexed levels per matrix travel as a second
// kernel parameter of the 8-bit kernels only, so the 3- and 4-bit launches keep
// their small parameter block.
struct Levels8 {
    uint16_t v[kMaxItems][256];
};
struct NoLevels {
    int32_t unused;
};
template <int BITS>
using LevelsT = typename std::conditional<BITS == 8, Levels8, NoLevels>::type;

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// Table entry at byte offset off from the table base.
__device__ __forceinline__ uint32_t lds_tab(uint32_t off)
{
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1+%2];" : "=r"(v) : "r"(off), "n"(kTabOff));
    return v;
}

template <int NW>
struct CodeVec { uint32_t w[NW]; };

template <int NW>
__device__ __forceinline__ CodeVec<NW> ld_codes(const uint8_t* p)
{
    CodeVec<NW> c;
    if constexpr (NW == 4) {
        asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                     : "=r"(c.w[0]), "=r"(c.w[1]), "=r"(c.w[2]), "=r"(c.w[3]) : "l"(p));
    } else if constexpr (NW == 2) {
        asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];"
                     : "=r"(c.w[0]), "=r"(c.w[1]) : "l"(p));
    } else {
#pragma unroll
        for (int i = 0; i < NW; ++i)
            asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(c.w[i]) : "l"(p + 4 * i));
    }
    return c;
}

template <bool F16>
__device__ __forceinline__ void fma_pair(float& a0, float& a1, uint32_t w, uint32_t x)
{
    if constexpr (F16) {
        asm("{.reg .b16 wl, wh, xl, xh;\n\t"
            "mov.b32 {wl, wh}, %2;\n\t"
            "mov.b32 {xl, xh}, %3;\n\t"
            "fma.rn.f32.f16 %0, wl, xl, %0;\n\t"
            "fma.rn.f32.f16 %1, wh, xh, %1;}"
            : "+f"(a0), "+f"(a1) : "r"(w), "r"(x));
    } else {
        asm("{.reg .b16 wl, wh, xl, xh;\n\t"
            "mov.b32 {wl, wh}, %2;\n\t"
            "mov.b32 {xl, xh}, %3;\n\t"
            "fma.rn.f32.bf16 %0, wl, xl, %0;\n\t"
            "fma.rn.f32.bf16 %1, wh, xh, %1;}"
            : "+f"(a0), "+f"(a1) : "r"(w), "r"(x));
    }
}

// 8-bit: two looked-up entries (each holding its 16-bit value in both halves)
// times one activation pair.
template <bool F16>
__device__ __forceinline__ void fma_two(float& a0, float& a1, uint32_t w0, uint32_t w1, uint32_t x)
{
    if constexpr (F16) {
        asm("{.reg .b16 al, ah, bl, bh, xl, xh;\n\t"
            "mov.b32 {al, ah}, %2;\n\t"
            "mov.b32 {bl, bh}, %3;\n\t"
            "mov.b32 {xl, xh}, %4;\n\t"
            "fma.rn.f32.f16 %0, al, xl, %0;\n\t"
            "fma.rn.f32.f16 %1, bl, xh, %1;}"
            : "+f"(a0), "+f"(a1) : "r"(w0), "r"(w1), "r"(x));
    } else {
        asm("{.reg .b16 al, ah, bl, bh, xl, xh;\n\t"
            "mov.b32 {al, ah}, %2;\n\t"
            "mov.b32 {bl, bh}, %3;\n\t"
            "mov.b32 {xl, xh}, %4;\n\t"
            "fma.rn.f32.bf16 %0, al, xl, %0;\n\t"
            "fma.rn.f32.bf16 %1, bl, xh, %1;}"
            : "+f"(a0), "+f"(a1) : "r"(w0), "r"(w1), "r"(x));
    }
}

// Reduce V per-lane values over the 32 lanes; afterwards lane l holds the
// total of value index (l >> (5 - log2 V)) in a[0] (V <= 32, power of two).
template <int V>
__device__ __forceinline__ void reduce_scatter(float (&a)[V], int lane)
{
    int count = V;
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        if (count > 1) {
            const int half = count / 2;
            const bool upper = (lane & m) != 0;
#pragma unroll
            for (int i = 0; i < V / 2; ++i) {
                if (i < half) {
                    const float send = upper ? a[i] : a[i + half];
                    const float keep = upper ? a[i + half] : a[i];
                    a[i] = keep + __shfl_xor_sync(0xffffffffu, send, m);
                }
            }
            count = half;
        } else {
            a[0] += __shfl_xor_sync(0xffffffffu, a[0], m);
        }
    }
}

__device__ __forceinline__ void store_y(void* Y, int dtype, int64_t idx, float v)
{
    if (dtype == LOGQ_F32) {
        static_cast<float*>(Y)[idx] = v;
    } else if (dtype == LOGQ_BF16) {
        static_cast<__nv_bfloat16*>(Y)[idx] = __float2bfloat16_rn(v);
    } else {
        static_cast<__half*>(Y)[idx] = __float2half_rn(v);
    }
}

// Table offsets of the four pair entries of one 4-bit code word: base_lane
// holds 4 * lane in byte 0 and zeros above, so one byte permute yields
// byte * 256 + 4 * lane.
__device__ __forceinline__ void addrs4(uint32_t c, uint32_t base_lane, uint32_t (&o)[4])
{
    o[0] = prmt(c, base_lane, 0x7604u);
    o[1] = prmt(c, base_lane, 0x7614u);
    o[2] = prmt(c, base_lane, 0x7624u);
    o[3] = prmt(c, base_lane, 0x7634u);
}

// Table offsets of the 16 pair entries of one 3-bit group (W0, W1, W2); the
// 6-bit field lands in bits 8-13, base_lane supplies 4 * lane.
__device__ __forceinline__ void addrs3(const uint32_t (&w)[3], uint32_t base_lane, uint32_t (&o)[16])
{
#pragma unroll
    for (int i = 0; i < 3; ++i) {
        o[5 * i + 0] = ((w[i] << 8) & 0x3f00u) | base_lane;
        o[5 * i + 1] = ((w[i] << 2) & 0x3f00u) | base_lane;
        o[5 * i + 2] = ((w[i] >> 4) & 0x3f00u) | base_lane;
        o[5 * i + 3] = ((w[i] >> 10) & 0x3f00u) | base_lane;
        o[5 * i + 4] = ((w[i] >> 16) & 0x3f00u) | base_lane;
    }
    o[15] = ((w[0] >> 22) & 0x0300u) | ((w[1] >> 20) & 0x0c00u) | ((w[2] >> 18) & 0x3000u) | base_lane;
}

// Decode one row's codes of this lane and accumulate B dot-product partials.
template <int BITS, int B, int NW, bool F16, int NPAIR>
__device__ __forceinline__ void decode_row(const CodeVec<NW>& c, uint32_t base_lane,
                                           const uint32_t (&xr)[B][NPAIR], float* acc, float* acc_hi)
{
    if constexpr (BITS == 8) {
        // word wi holds the codes of k = 4 wi .. 4 wi + 3, one per byte
#pragma unroll
        for (int wi = 0; wi < NW; ++wi) {
            uint32_t o[4];
            addrs4(c.w[wi], base_lane, o);
            const uint32_t v0 = lds_tab(o[0]), v1 = lds_tab(o[1]), v2 = lds_tab(o[2]), v3 = lds_tab(o[3]);
#pragma unroll
            for (int b = 0; b < B; ++b) {
                fma_two<F16>(acc[b], acc_hi[b], v0, v1, xr[b][2 * wi]);
                fma_two<F16>(acc[b], acc_hi[b], v2, v3, xr[b][2 * wi + 1]);
            }
        }
    } else if constexpr (BITS == 4) {
#pragma unroll
        for (int wi = 0; wi < NW; ++wi) {
            uint32_t o[4];
            addrs4(c.w[wi], base_lane, o);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint32_t wp = lds_tab(o[j]);
#pragma unroll
                for (int b = 0; b < B; ++b) fma_pair<F16>(acc[b], acc_hi[b], wp, xr[b][4 * wi + j]);
            }
        }
    } else {
#pragma unroll
        for (int gi = 0; gi < NW / 3; ++gi) {
            uint32_t o[16];
            const uint32_t w3[3] = {c.w[3 * gi], c.w[3 * gi + 1], c.w[3 * gi + 2]};
            addrs3(w3, base_lane, o);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const uint32_t wp = lds_tab(o[j]);
#pragma unroll
                for (int b = 0; b < B; ++b) fma_pair<F16>(acc[b], acc_hi[b], wp, xr[b][16 * gi + j]);
            }
        }
    }
}

template <int BITS, int B, int KW, int R, bool F16, int NT, int MINB = 512 / NT>
__global__ void __launch_bounds__(NT, MINB) gemv_kernel(const __grid_constant__ GemvParams p,
                                                            const __grid_constant__ LevelsT<BITS> lv)
{
    extern __shared__ __align__(16) uint8_t smem[];
    constexpr int NPAIR = KW / 2;                            // bf16 pairs of x per lane and batch row
    constexpr int NW = (BITS == 8) ? KW / 4 : (BITS == 4) ? KW / 8 : 3 * KW / 32;   // code words per lane and row
    constexpr int NENT = (BITS == 3) ? 64 : 256;
    constexpr uint32_t TAB_BYTES = NENT * kTabStride;
    constexpr int V = R * B;
    constexpr int SPAN = 32 * KW;
    static_assert(V <= 32 && (V & (V - 1)) == 0, "values per lane must be a power of two <= 32");

    // programmatic dependent launch: the next kernel on the stream may start
    // now.  Its CTAs may run beside this one and do their own prologue
    // meanwhile; they wait for this grid to finish before they touch X or Y.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if ((uint32_t)__cvta_generic_to_shared(smem) != kTabOff) {   // table addressing relies on it
        if (tid == 0) atomicExch(p.err, (uint32_t)LOGQ_ERR_UNSUPPORTED);
        return;
    }
    // this CTA's matrix and its contiguous range of rows
    int m = 0;
#pragma unroll
    for (int i = 1; i < kMaxItems; ++i)
        if (i < p.nitems && (int)blockIdx.x >= p.item[i].cta_begin) m = i;
    const GemvItem& item = p.item[m];
    const int c = (int)blockIdx.x - item.cta_begin;
    const int64_t r0 = (int64_t)c * item.rows_q + (c < item.rows_rem ? c : item.rows_rem);
    const int64_t r1 = r0 + item.rows_q + (c < item.rows_rem ? 1 : 0);

    // 0) the first round of code loads of this warp's first (chunk, span) goes
    //    out first: its latency hides behind the prologue below.  Codes are
    //    weights, not the previous kernel's output (see the launch contract).
    const int G = p.groups, SC = p.span_cols;
    const bool compute_warp = warp < G * SC;
    const int g = warp % G, scol = warp / G;
    const int64_t rstride = (int64_t)G * p.row_bytes;
    CodeVec<NW> ca[R], cb[R];
    auto span_first = [&](int64_t q0, int s, int& k0, bool& active) -> const uint8_t* {
        k0 = s * SPAN + lane * KW;
        active = k0 < p.K;
        // idle lanes read the row start (valid memory) and multiply by zero
        const int64_t lane_byte =
            active ? ((BITS == 8) ? (int64_t)k0 : (BITS == 4) ? (int64_t)k0 / 2 : (int64_t)k0 / 32 * 12) : 0;
        return item.codes + (q0 + g) * p.row_bytes + lane_byte;
    };
    // codes of the round whose first row is at rp, here = rows left from it
    auto load_round = [&](CodeVec<NW> (&c)[R], const uint8_t* rp, int here) {
        if (here >= R) {
#pragma unroll
            for (int r = 0; r < R; ++r) c[r] = ld_codes<NW>(rp + r * rstride);
        } else {
#pragma unroll
            for (int r = 0; r < R; ++r)
                if (r < here) c[r] = ld_codes<NW>(rp + r * rstride);
        }
    };
    bool preloaded = false;                     // ca holds the first round of the first (chunk, span)
    {
        const int nrows0 = (int)((r0 + p.chunk_rows < r1 ? r0 + p.chunk_rows : r1) - r0);
        const int my_rows0 = (nrows0 > g) ? (nrows0 - g + G - 1) / G : 0;
        if (compute_warp && my_rows0 > 0 && scol < p.spans) {
            int k0;
            bool active;
            load_round(ca, span_first(r0, scol, k0, active), my_rows0);
            preloaded = true;
        }
    }

    // 1) start streaming this CTA's code rows into L2, and its share of the
    //    optional warm-up range.
    {
        constexpr int64_t piece = 16384;
        const uint8_t* base = item.codes + r0 * p.row_bytes;
        int64_t bytes = p.own_pf ? (r1 - r0) * p.row_bytes : 0;
        if (bytes > kPrefetchCap) bytes = kPrefetchCap;
        for (int64_t off = (int64_t)tid * piece; off < bytes; off += (int64_t)NT * piece) {
            const int64_t n = (bytes - off) < piece ? (bytes - off) : piece;
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base + off), "r"((uint32_t)n)
                         : "memory");
        }
        if (p.pf_bytes > 0) {
            const int64_t beg = p.pf_share * blockIdx.x;
            const int64_t end = (beg + p.pf_share < p.pf_bytes) ? beg + p.pf_share : p.pf_bytes;
            for (int64_t off = beg + (int64_t)tid * piece; off < end; off += (int64_t)NT * piece) {
                const int64_t n = (end - off) < piece ? (end - off) : piece;
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p.pf + off), "r"((uint32_t)n)
                             : "memory");
            }
        }
    }

    // 2) pair table: entry e = (value of its low code) | (value of its high
    //    code) << 16, 32 copies (one per lane) in the first 128 bytes of its
    //    256-byte row.  The 16 levels are staged in the free half of row 0
    //    (indexed parameter reads with per-thread indices would serialise).
    //    8-bit codes: entry e is the value of code e in both halves.
    if constexpr (BITS == 8) {
        for (int i = tid; i < NENT * 8; i += NT) {
            const int e = i >> 3, part = i & 7;
            const uint32_t v = (uint32_t)lv.v[m][e] * 0x10001u;
            reinterpret_cast<uint4*>(smem + e * kTabStride)[part] = make_uint4(v, v, v, v);
        }
    } else {
        uint32_t* lvl = reinterpret_cast<uint32_t*>(smem + kLvlOff);
        if (tid < 16) lvl[tid] = item.lvl16[tid] & 0xffffu;
        __syncthreads();
        for (int i = tid; i < NENT * 8; i += NT) {
            const int e = i >> 3, part = i & 7;
            const uint32_t lo = (BITS == 4) ? (e & 15) : (e & 7);
            const uint32_t hi = (BITS == 4) ? (e >> 4) : (e >> 3);
            const uint32_t v = lvl[lo] | (lvl[hi] << 16);
            reinterpret_cast<uint4*>(smem + e * kTabStride)[part] = make_uint4(v, v, v, v);
        }
    }
    // span partial i (in the free half of table row i / 32, or after the table)
    auto red = [&](int i) -> float& {
        if constexpr (red_in_table(BITS, B))
            return *reinterpret_cast<float*>(smem + (i >> 5) * kTabStride + 128 + (i & 31) * 4);
        else
            return reinterpret_cast<float*>(smem + TAB_BYTES)[i];
    };
    __syncthreads();

    const uint32_t base_lane = 4u * (uint32_t)lane;
    constexpr int lg2V = (V >= 32) ? 5 : (V >= 16) ? 4 : (V >= 8) ? 3 : (V >= 4) ? 2 : (V >= 2) ? 1 : 0;
    const int my_v = lane >> (5 - lg2V);
    const bool writer = (lane & ((32 >> lg2V) - 1)) == 0;

    for (int64_t q0 = r0; q0 < r1; q0 += p.chunk_rows) {
        const int64_t q1 = (q0 + p.chunk_rows < r1) ? q0 + p.chunk_rows : r1;
        const int nrows = (int)(q1 - q0);
        const int my_rows = (nrows > g) ? (nrows - g + G - 1) / G : 0;
        if (compute_warp && my_rows > 0) {
            for (int s = scol; s < p.spans; s += SC) {
                int k0;
                bool active;
                const uint8_t* first = span_first(q0, s, k0, active);
                // Rounds of R rows with two code buffers: the loads of round t+1 are
                // in flight while round t is decoded.  Full rounds run unguarded;
                // the last round guards its rows (warp-uniform branches).
                if (!preloaded) load_round(ca, first, my_rows);
                preloaded = false;
                asm volatile("griddepcontrol.wait;" ::: "memory");
                // activations for this span stay in registers (zero on idle lanes)
                uint32_t xr[B][NPAIR];
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const uint16_t* xp = p.X + (int64_t)b * p.K + (active ? k0 : 0);
#pragma unroll
                    for (int i = 0; i < NPAIR; i += 4) {
                        uint4 v = make_uint4(0, 0, 0, 0);
                        if (active && b < p.B) v = *reinterpret_cast<const uint4*>(xp + 2 * i);
                        xr[b][i] = v.x;
                        if (i + 1 < NPAIR) xr[b][i + 1] = v.y;
                        if (i + 2 < NPAIR) xr[b][i + 2] = v.z;
                        if (i + 3 < NPAIR) xr[b][i + 3] = v.w;
                    }
                }
                // the writer lane's result of each round: row my_v / B, batch
                // row my_v % B; its local row and partial-buffer index advance
                // by constants
                int lr_w = g + G * (my_v / B);
                int red_i = (s * p.chunk_rows + lr_w) * B + my_v % B;
                auto run_round = [&](const CodeVec<NW> (&c)[R], int here) {
                    float acc[V], acc_hi[V];
#pragma unroll
                    for (int i = 0; i < V; ++i) acc[i] = acc_hi[i] = 0.f;
                    if (here >= R) {
#pragma unroll
                        for (int r = 0; r < R; ++r) decode_row<BITS, B, NW, F16>(c[r], base_lane, xr, acc + r * B, acc_hi + r * B);
                    } else {
#pragma unroll
                        for (int r = 0; r < R; ++r)
                            if (r < here) decode_row<BITS, B, NW, F16>(c[r], base_lane, xr, acc + r * B, acc_hi + r * B);
                    }
#pragma unroll
                    for (int i = 0; i < V; ++i) acc[i] += acc_hi[i];
                    reduce_scatter<V>(acc, lane);
                    if (writer && lr_w < nrows) red(red_i) = acc[0];
                    lr_w += G * R;
                    red_i += G * R * B;
                };
                // rounds of R rows with two code buffers: the loads of the next
                // round are in flight while this one is decoded
                if constexpr (R == 1) {
                    // one-row rounds (batches of 8 and 16): a counted loop with
                    // indices recomputed from the round number, which keeps
                    // fewer registers live in these register-bound kernels
                    auto load1 = [&](CodeVec<NW> (&c)[R], int t) {
                        if (t < my_rows) c[0] = ld_codes<NW>(first + (int64_t)t * rstride);
                    };
                    auto run1 = [&](const CodeVec<NW> (&c)[R], int t) {
                        float acc[V], acc_hi[V];
#pragma unroll
                        for (int i = 0; i < V; ++i) acc[i] = acc_hi[i] = 0.f;
                        if (t < my_rows) decode_row<BITS, B, NW, F16>(c[0], base_lane, xr, acc, acc_hi);
#pragma unroll
                        for (int i = 0; i < V; ++i) acc[i] += acc_hi[i];
                        reduce_scatter<V>(acc, lane);
                        if (writer) {
                            const int lr = g + G * t;
                            if (lr < nrows) red((s * p.chunk_rows + lr) * B + my_v % B) = acc[0];
                        }
                    };
                    const int nrounds = my_rows;
                    for (int t = 0; t < nrounds; t += 2) {
                        load1(cb, t + 1);
                        run1(ca, t);
                        if (t + 1 >= nrounds) break;
                        load1(ca, t + 2);
                        run1(cb, t + 1);
                    }
                } else {
                    // Full rounds run without any row checks (branches and their
                    // convergence points were a quarter of the loop's
                    // instructions); only the last, partial round checks its rows.
                    // ca holds round 0 (full, or the partial round itself).
                    const int nfull = my_rows / R, tail = my_rows - nfull * R;
                    const int64_t rstep = (int64_t)R * rstride;
                    auto load_full = [&](CodeVec<NW> (&c)[R], const uint8_t* rp) {
#pragma unroll
                        for (int r = 0; r < R; ++r) c[r] = ld_codes<NW>(rp + r * rstride);
                    };
                    auto run_full = [&](const CodeVec<NW> (&c)[R]) {
                        float acc[V], acc_hi[V];
#pragma unroll
                        for (int i = 0; i < V; ++i) acc[i] = acc_hi[i] = 0.f;
#pragma unroll
                        for (int r = 0; r < R; ++r)
                            decode_row<BITS, B, NW, F16>(c[r], base_lane, xr, acc + r * B, acc_hi + r * B);
#pragma unroll
                        for (int i = 0; i < V; ++i) acc[i] += acc_hi[i];
                        reduce_scatter<V>(acc, lane);
                        if (writer) red(red_i) = acc[0];            // a full round's rows all exist
                        lr_w += G * R;
                        red_i += G * R * B;
                    };
                    const uint8_t* rp = first;
                    int t = 0;
                    for (; t + 2 <= nfull; t += 2) {                // rounds t (in ca) and t + 1
                        load_full(cb, rp + rstep);
                        run_full(ca);
                        if (t + 2 < nfull) load_full(ca, rp + 2 * rstep);
                        else if (tail) load_round(ca, rp + 2 * rstep, tail);
                        run_full(cb);
                        rp += 2 * rstep;
                    }
                    if (t < nfull) {                                 // one full round left, in ca
                        if (tail) load_round(cb, rp + rstep, tail);
                        run_full(ca);
                        if (tail) run_round(cb, tail);
                    } else if (tail) {
                        run_round(ca, tail);
                    }
                }
            }
        }
        asm volatile("griddepcontrol.wait;" ::: "memory");
        __syncthreads();
        // fixed-order sum over spans
        for (int i = tid; i < nrows * B; i += NT) {
            const int lr = i / B, b = i % B;
            if (b >= p.B) continue;
            float sum = 0.f;
            for (int s = 0; s < p.spans; ++s) sum += red((s * p.chunk_rows + lr) * B + b);
            store_y(item.Y, p.y_dtype, (int64_t)b * item.N + q0 + lr, sum);
        }
        __syncthreads();
    }
}

struct Config {
    int bits, B, KW, R;
};

// Dynamic shared memory opt-in and a carveout that leaves room for two CTAs
// per SM: per-device function attributes, set once per device.
template <int BITS, int B, int KW, int R, bool F16, int NT, int MINB = 512 / NT>
cudaError_t run(const GemvParams& p, const GroupArgs& a, int grid, size_t smem, cudaStream_t s)
{
    LevelsT<BITS> lv;
    memset(&lv, 0, sizeof lv);
    if constexpr (BITS == 8)
        for (int i = 0; i < a.count; ++i)
            for (int c = 0; c < 256; ++c) lv.v[i][c] = a.item[i].lvl16[c];
    auto k = gemv_kernel<BITS, B, KW, R, F16, NT, MINB>;
    static bool configured[64] = {false};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                                 B <= 2 ? LOGQ_GEMV_CARVEOUT : (int)cudaSharedmemCarveoutMaxShared);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(NT);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k, p, lv);
}

template <bool F16>
cudaError_t dispatch(int bits, int Bp, bool large, bool tiny, const GemvParams& p, const GroupArgs& a, int grid,
                     size_t smem, cudaStream_t s)
{
    constexpr int L = kLargeThreads, S = kSmallThreads;
    if (bits == 8) {
        switch (Bp) {
        case 1: return large ? run<8, 1, 16, 8, F16, L>(p, a, grid, smem, s) : run<8, 1, 16, 8, F16, S>(p, a, grid, smem, s);
        case 2: return large ? run<8, 2, 16, 4, F16, L>(p, a, grid, smem, s) : run<8, 2, 16, 4, F16, S>(p, a, grid, smem, s);
        case 4: return run<8, 4, 16, 2, F16, S>(p, a, grid, smem, s);
        }
    } else if (bits == 4) {
        switch (Bp) {
        // batch 1: 8-warp CTAs, two per SM (tiny launches: one per SM)
        case 1:
            return tiny ? run<4, 1, 16, 8, F16, S, kTinyPerSm>(p, a, grid, smem, s)
                        : run<4, 1, 32, 8, F16, S, 2>(p, a, grid, smem, s);
        case 2: return large ? run<4, 2, 32, 4, F16, L>(p, a, grid, smem, s) : run<4, 2, 32, 4, F16, S>(p, a, grid, smem, s);
        // batch 4: large launches one 16-warp CTA per SM with 32 k per lane,
        // small ones two 8-warp CTAs with 16 k; batch 8 one 16-warp CTA with
        // 16 k; batch 16 one 8-warp CTA whose threads hold 16 k of all 16
        // activation rows (251 registers)
        case 4: return large ? run<4, 4, 32, 2, F16, L, 1>(p, a, grid, smem, s)
                             : run<4, 4, 16, 2, F16, S>(p, a, grid, smem, s);
        case 8: return run<4, 8, 16, 1, F16, L, 1>(p, a, grid, smem, s);
        case 16: return run<4, 16, 16, 1, F16, S, 1>(p, a, grid, smem, s);
        }
    } else {
        switch (Bp) {
        case 1: return large ? run<3, 1, 32, 8, F16, L>(p, a, grid, smem, s) : run<3, 1, 32, 8, F16, S>(p, a, grid, smem, s);
        case 2: return large ? run<3, 2, 32, 4, F16, L>(p, a, grid, smem, s) : run<3, 2, 32, 4, F16, S>(p, a, grid, smem, s);
        case 4: return run<3, 4, 32, 2, F16, S>(p, a, grid, smem, s);
        }
    }
    return cudaErrorInvalidValue;
}

int padded_batch(int64_t B)
{
    if (B <= 1) return 1;
    if (B <= 2) return 2;
    if (B <= 4) return 4;
    if (B <= 8) return 8;
    return 16;
}

int kw_for(int bits, int Bp, bool tiny, bool large)
{
    if (bits == 8) return 16;
    if (bits == 3) return 32;
    if (Bp == 1 && tiny) return 16;
    if (Bp <= 2) return 32;
    if (Bp == 4) return large ? 32 : 16;
    return 16;
}

// The table lookups address shared memory relative to kTabOff, which is where
// dynamic shared memory starts when a kernel has no static shared memory.
cudaError_t check_shared_base()
{
    static int ok[64] = {0};   // 0 unknown, 1 yes, -1 no
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (ok[dev] == 0) {
        int reserved = -1;
        e = cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
        if (e != cudaSuccess) return e;
        ok[dev] = (reserved == (int)kTabOff) ? 1 : -1;
    }
    return ok[dev] > 0 ? cudaSuccess : cudaErrorNotSupported;
}

}  // namespace

bool gemv_supports(int bits, int64_t B)
{
    if (bits == 4) return B >= 1 && B <= 16;
    if (bits == 3 || bits == 8) return B >= 1 && B <= 4;
    return false;
}

cudaError_t launch_gemv_group(const GroupArgs& a, cudaStream_t s)
{
    if (a.count < 1 || a.count > kMaxItems) return cudaErrorInvalidValue;
    cudaError_t e = check_shared_base();
    if (e != cudaSuccess) return e;
    const int Bp = padded_batch(a.B);
    int64_t total_rows = 0;
    for (int i = 0; i < a.count; ++i) total_rows += a.item[i].N;
    const int64_t row_bytes = (a.bits == 8) ? a.K : (a.bits == 4) ? a.K / 2 : a.K / 32 * 12;
    const bool tiny = a.bits == 4 && Bp == 1 && total_rows * row_bytes < kTinyBytes;
    // large launches: batch 1-2 (and 4-bit batch 4) with at least kSplitBytes of codes
    const bool large = (Bp <= 2 || (a.bits == 4 && Bp == 4)) && total_rows * row_bytes >= kSplitBytes;
    const int KW = kw_for(a.bits, Bp, tiny, large);
    const int span = 32 * KW;
    GemvParams p;
    memset(&p, 0, sizeof p);
    p.nitems = a.count;
    p.X = static_cast<const uint16_t*>(a.X);
    p.err = &a.ws->error;
    p.K = (int32_t)a.K;
    p.B = (int32_t)a.B;
    p.y_dtype = a.y_dtype;
    p.row_bytes = row_bytes;
    p.spans = (int32_t)((a.K + span - 1) / span);
    // Batch 1-2: large launches one 512-thread CTA per SM, small ones one
    // 256-thread CTA per SM.  3- and 8-bit batch 4: two 256-thread CTAs per SM;
    // 4-bit batches of 4 and more: see dispatch() for the shapes.
    const bool wide4 = a.bits == 4 && ((Bp == 4 && large) || Bp == 8);
    const bool b1_4 = a.bits == 4 && Bp == 1;
    const int threads = ((large && !b1_4) || wide4) ? kLargeThreads : kSmallThreads;
    const int per_sm = b1_4 ? (tiny ? kTinyPerSm : 2)
                            : (Bp >= 4 && !(a.bits == 4 && (Bp >= 8 || large))) ? 2 : 1;
    const int warps = threads / 32;
    if (p.spans >= warps) {
        p.groups = 1;
        p.span_cols = warps;
    } else {
        p.groups = warps / p.spans;
        p.span_cols = p.spans;
    }
    // Each CTA's own rows are prefetched into L2 up front only where that was
    // measured to pay: not in 4-bit batch-1 launches (two CTAs per SM, whose
    // code loads keep enough in flight) except tiny ones, nor in large launches.
    p.own_pf = b1_4 ? (tiny ? LOGQ_GEMV_TINY_OWN_PF : 0) : (large ? 0 : 1);
    // The warm-up range is prefetched only when it is below kSplitBytes: a
    // launch that large streams its own codes at full rate, and warming L2
    // with them slows the launch that issues the prefetch more than it helps.
    p.pf = static_cast<const uint8_t*>(a.pf);
    p.pf_bytes = (a.pf && a.pf_bytes < kSplitBytes) ? a.pf_bytes : 0;

    // CTAs in proportion to each matrix's rows (at least one each, at most one
    // per row).
    const int sms = sm_count() > 0 ? sm_count() : 148;
    int grid = (int)(total_rows < (int64_t)sms * per_sm ? total_rows : (int64_t)sms * per_sm);
    if (grid < a.count) grid = a.count;
    int ctas[kMaxItems] = {0};
    int used = 0;
    for (int i = 0; i < a.count; ++i) {
        int64_t c = (int64_t)grid * a.item[i].N / total_rows;
        if (c < 1) c = 1;
        if (c > a.item[i].N) c = a.item[i].N;
        ctas[i] = (int)c;
        used += ctas[i];
    }
    while (used < grid) {               // hand out what rounding left, largest rows per CTA first
        int best = -1;
        double best_load = -1.0;
        for (int i = 0; i < a.count; ++i) {
            if (ctas[i] >= a.item[i].N) continue;
            const double load = (double)a.item[i].N / ctas[i];
            if (load > best_load) { best_load = load; best = i; }
        }
        if (best < 0) break;
        ++ctas[best];
        ++used;
    }
    while (used > grid) {               // too many (minimums): take from the lightest
        int best = -1;
        double best_load = 1e300;
        for (int i = 0; i < a.count; ++i) {
            if (ctas[i] <= 1) continue;
            const double load = (double)a.item[i].N / ctas[i];
            if (load < best_load) { best_load = load; best = i; }
        }
        if (best < 0) break;
        --ctas[best];
        --used;
    }
    grid = used;
    p.pf_share = p.pf_bytes > 0 ? (((p.pf_bytes + grid - 1) / grid + 15) & ~(int64_t)15) : 0;
    int64_t max_rows = 0;
    int begin = 0;
    for (int i = 0; i < a.count; ++i) {
        GemvItem& it = p.item[i];
        it.codes = a.item[i].codes;
        it.Y = a.item[i].Y;
        it.N = (int32_t)a.item[i].N;
        it.cta_begin = begin;
        it.cta_count = ctas[i];
        it.rows_q = (int32_t)(a.item[i].N / ctas[i]);
        it.rows_rem = (int32_t)(a.item[i].N % ctas[i]);
        for (int c = 0; c < 16; ++c) it.lvl16[c] = a.item[i].lvl16[c];
        begin += ctas[i];
        const int64_t rows = it.rows_q + (it.rows_rem ? 1 : 0);
        if (rows > max_rows) max_rows = rows;
    }
    int64_t chunk = kRedBytes / ((int64_t)p.spans * Bp * 4);
    if (chunk > max_rows) chunk = max_rows;
    if (chunk < 1) return cudaErrorInvalidValue;
    p.chunk_rows = (int32_t)chunk;
    const size_t tab = (size_t)(a.bits == 3 ? 64 : 256) * kTabStride;
    const size_t smem = red_in_table(a.bits, Bp) ? tab : tab + (size_t)p.spans * chunk * Bp * 4;
    return a.x_f16 ? dispatch<true>(a.bits, Bp, large, tiny, p, a, grid, smem, s)
                   : dispatch<false>(a.bits, Bp, large, tiny, p, a, grid, smem, s);
}

cudaError_t launch_gemv(const LinearArgs& a, cudaStream_t s)
{
    GroupArgs g;
    memset(&g, 0, sizeof g);
    g.count = 1;
    g.item[0].codes = a.codes;
    g.item[0].Y = a.Y;
    g.item[0].N = a.N;
    for (int c = 0; c < 256; ++c) g.item[0].lvl16[c] = a.lvl16[c];
    g.X = a.X;
    g.B = a.B;
    g.K = a.K;
    g.bits = a.bits;
    g.x_f16 = a.x_f16;
    g.y_dtype = a.y_dtype;
    g.ws = a.ws;
    return launch_gemv_group(g, s);
}

}  // namespace logq
