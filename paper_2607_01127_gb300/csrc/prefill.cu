// Prefill GEMM on the tensor cores: Y[t][n] = sum_k X[t][k] * table[code(n, k)]
// (paper Sec. 3.3; the paper attributes its large-batch slowdown to per-element
// LUT reads, so here each weight is dequantised once per tile and reused by a
// dense bf16/fp16 contraction).
//
// One persistent CTA per SM walks 128 (weights) x BN (tokens) output tiles, BN
// = 256 for prefill and 16 for small batches; where there are too few tiles
// to fill the SMs, each tile's k range is split into ranges taken by
// different CTAs, which write fp32 partial sums to the caller's workspace and
// a second kernel adds them in a fixed order.  A launch may cover up to four
// matrices that read the same X (q/k/v, gate/up): each gets a contiguous
// range of the CTAs, in proportion to its tiles, and a CTA works on its
// matrix's tiles only.
// The dequantised weight tile (the MMA's A operand) lives in tensor memory, not
// in shared memory: tensor memory holds one fp32 accumulator (256 columns) and
// eight weight stages (32 columns each), and shared memory holds the pair table
// and five X stages.
// Warp roles:
//   warp 0     TMA producer: X tiles [256 tokens x 64 k] with 128-byte swizzle.
//   warp 1     MMA issuer: tcgen05.mma kind::f16, M = 128 (weight rows),
//              N = 256 (tokens), K = 16, A from tensor memory, B (X) from
//              shared memory, fp32 accumulator in tensor memory.  Also
//              allocates TMEM.
//   warps 2-9  epilogue: two warps per TMEM lane quarter, each draining 128
//              token columns with tcgen05.ld; 16-bit outputs are rounded into
//              registers and the accumulator is handed back before the stores
//              of Y (lane n writes Y[t][n0 + n]).
//   warps 10-17 decode: two threads per weight row of the tile, each owning 32
//              of the stage's 64 k; a thread streams its codes into its own
//              16-byte slot of a shared ring with cp.async, resolves two codes
//              per lookup in a per-lane-replicated pair table, and writes the
//              16 bf16 (or fp16) pairs to its row's TMEM lane with tcgen05.st.
//              tcgen05.st reaches only the warp's lane quarter (warp % 4), so a
//              thread's weight row is 32 * (warp % 4) + lane.
// The pair table starts the dynamic shared memory, at the fixed shared address
// kTabOff, with 256-byte rows: the offset of an entry, byte << 8 | 4 * lane,
// is one byte permute of the code word and the table base is the load's
// immediate offset.  The code ring lives in the free upper halves of the rows.
// Every mbarrier wait is bounded: a wait that exceeds ~1 s of clock cycles
// raises an abort flag, records LOGQ_ERR_TIMEOUT in the caller's workspace and
// lets every role leave its loop; the kernel drains what it issued, frees its
// tensor memory and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>
#include <stdint.h>
#include <string.h>

#include <mutex>

#include "internal.h"

namespace logq {
namespace {

constexpr int kBM = 128;                 // weight rows per tile (MMA M)
constexpr int kBNMax = 256;              // widest token tile (MMA N)
constexpr int kBK = 64;                  // k per stage (one 128-byte swizzle atom of bf16)
constexpr int kMaxPrefillItems = 4;      // matrices of one grouped launch
constexpr int kXStages = 5;              // X tiles in flight (TMA)
constexpr int kWStages = 8;              // dequantised weight tiles in flight (tensor memory)
// Decode warps: four per k slice of a stage (one per TMEM lane quarter), each
// thread owning one weight row's kSliceK of the stage's 64 k.  Eight (two
// slices of 32 k) measured faster than sixteen (four of 16 k, 72 registers):
// the per-stage waits, tensor-memory store and arrive of each warp cost more
// than the extra warps hide.
#ifndef LOGQ_PREFILL_DECODE_WARPS
#define LOGQ_PREFILL_DECODE_WARPS 8
#endif
constexpr int kDecodeWarps = LOGQ_PREFILL_DECODE_WARPS;
static_assert(kDecodeWarps == 4 || kDecodeWarps == 8 || kDecodeWarps == 16, "one, two or four k slices per stage");
constexpr int kSlices = kDecodeWarps / 4;
constexpr int kSliceK = 64 / kSlices;            // k per decode thread and stage: 64, 32 or 16
constexpr int kSlicePairs = kSliceK / 2;         // TMEM columns (16-bit pairs) per thread and stage
constexpr int kDecodeThreads = 32 * kDecodeWarps;
constexpr int kEpiWarps = 8;                       // two per TMEM lane quarter
constexpr int kEpi0 = 2, kDec0 = kEpi0 + kEpiWarps;  // first epilogue / decode warp
constexpr int kThreads = 32 * (kDec0 + kDecodeWarps);  // producer, MMA, epilogue, decode
constexpr int kCodeSlotBytes = 16;               // ring slot: codes of one thread's slice (<= 16 B)
constexpr int kCodeStageBytes = kDecodeThreads * kCodeSlotBytes;
// Shared address at which dynamic shared memory starts in a kernel without
// static shared memory (the per-CTA reserved area comes first).
constexpr uint32_t kTabOff = 1024;
constexpr uint32_t kTabRow = 256;                // 32 lane copies in the first 128 bytes
constexpr uint32_t kTabRegion = 256 * kTabRow;   // table rows (the 4-bit table uses all 256)
constexpr uint32_t kTmemCols = 512;              // accumulator (256) + weight stages (8 x 32)
constexpr uint32_t kWCol0 = kBNMax;              // first column of weight stage 0 (after the widest accumulator)
constexpr uint32_t kWStageCols = kBK / 2;        // 64 k of 16-bit values = 32 columns
static_assert(kWCol0 + kWStages * kWStageCols <= kTmemCols, "weight stages must fit in tensor memory");
constexpr long long kWaitLimit = 2000000000LL;   // cycles (~1 s)

// error detail codes (workspace->detail)
enum : uint32_t { kWaitProducer = 1, kWaitMma = 2, kWaitEpilogue = 3, kWaitDecode = 4, kWaitDrain = 5,
                  kWaitLayout = 6 };
#ifdef LOGQ_TEST_WAIT_HOOK
constexpr uint32_t kTestStallWord = 0x57A11u;   // workspace reserved[0] value that triggers the test stall
#endif

// One matrix of a launch.  A grouped launch (matrices sharing X) gives each
// matrix a contiguous range of CTAs, in proportion to its tiles; a CTA works
// on its matrix's tiles only, so it builds one pair table.
struct PrefillItem {
    const uint8_t* codes;
    void* Y;
    float* part;            // splits > 1: fp32 partial sums [splits][B][N] (caller's workspace)
    int64_t N;
    int32_t n_tiles_n;
    int32_t cta_begin;      // first CTA of this matrix
    int32_t ncta;           // its CTAs
    int32_t pad_;
    uint16_t lvl16[256];    // code-indexed 16-bit levels (2^bits used)
};

struct PrefillParams {
    PrefillItem item[kMaxPrefillItems];
    int32_t nitems;
    Workspace* ws;
    int32_t K, B;
    int64_t row_bytes;
    int32_t bits;
    int32_t y_dtype;
    int32_t n_tiles_t;
    int32_t splits;         // k ranges per output tile (the same for every matrix)
    int32_t ksplit;         // k-steps per range (the last may be shorter)
    uint32_t idesc;
    uint32_t smem_bytes;    // dynamic shared memory of the launch (layout check)
};

// ------------------------------------------------------------------ PTX ---

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait, slow path: polls until the phase completes, the abort flag
// rises (unless draining) or ~1 s of cycles pass; running out raises the
// abort flag and records LOGQ_ERR_TIMEOUT in the workspace.
__device__ __noinline__ bool wait_slow(uint32_t bar, uint32_t parity, volatile int* abort_flag, Workspace* ws,
                                       uint32_t who, bool drain)
{
    const long long t0 = clock64();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (!drain && *abort_flag) return false;
        if (clock64() - t0 > kWaitLimit) {
            *abort_flag = 1;
            atomicExch(&ws->detail, who);
            atomicExch(&ws->error, (uint32_t)LOGQ_ERR_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ bool wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                             Workspace* ws, uint32_t who, bool drain = false)
{
    if (mbar_try_wait(bar, parity)) return true;
    return wait_slow(bar, parity, abort_flag, ws, who, drain);
}

// One lane of the warp, chosen by the hardware; the rest of the warp keeps the
// same (uniform) control flow and operands.
__device__ __forceinline__ bool elect_one()
{
    uint32_t pred;
    asm volatile(
        "{\n\t.reg .pred P;\n\t.reg .b32 R;\n\t"
        "elect.sync R|P, 0xffffffff;\n\t"
        "selp.u32 %0, 1, 0, P;\n\t}"
        : "=r"(pred));
    return pred != 0;
}

// One lane of the warp polls (a barrier polled by many threads serialises);
// the outcome is broadcast to the whole warp.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag, Workspace* ws,
                                          uint32_t who)
{
    uint32_t ok = 0;
    if ((threadIdx.x & 31) == 0) ok = wait_bounded(bar, parity, abort_flag, ws, who) ? 1u : 0u;
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(dst), "l"(map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void cp_async_4(uint32_t dst, const void* src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_8(uint32_t dst, const void* src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row groups 1024 bytes apart (stride byte offset), version 1.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr)
{
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3ffffu) >> 4);          // start address
    d |= (uint64_t)1 << 16;                            // leading byte offset (unused for this layout)
    d |= (uint64_t)(1024 >> 4) << 32;                  // stride byte offset
    d |= (uint64_t)1 << 46;                            // descriptor version
    d |= (uint64_t)2 << 61;                            // swizzle: 128 bytes
    return d;
}

// A (weights) from tensor memory: row m in lane m, 16-bit k-pairs packed per column.
__device__ __forceinline__ void mma_f16_ta(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
        ::"r"(tmem_d), "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// 16 consecutive columns of this warp's 32 TMEM lanes (lane i of the warp -> TMEM lane base + i).
[[maybe_unused]] __device__ __forceinline__ void tmem_st_pairs(uint32_t taddr, const uint32_t (&v)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
        ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
          "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}

[[maybe_unused]] __device__ __forceinline__ void tmem_st_pairs(uint32_t taddr, const uint32_t (&v)[32])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
        ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
          "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]),
          "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]),
          "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
}

[[maybe_unused]] __device__ __forceinline__ void tmem_st_pairs(uint32_t taddr, const uint32_t (&v)[8])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
        ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
        : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void mma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Pair-table entry at byte offset off from the table base.
__device__ __forceinline__ uint32_t lds_tab(uint32_t off)
{
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1+%2];" : "=r"(v) : "r"(off), "n"(kTabOff));
    return v;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr)
{
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
                 : "memory");
}

// ------------------------------------------------------------------ kernel ---

// EIGHT: 8-bit codes, one per byte: a thread's kSliceK k of a stage are
// kSliceK bytes (one or two ring slots), each byte resolves to one value (the
// table holds it in both halves) and two values form a pair with one byte
// permute.
template <bool EIGHT, int BN>
__global__ void __launch_bounds__(kThreads, 1)
prefill_kernel(const __grid_constant__ PrefillParams p, const __grid_constant__ CUtensorMap xmap)
{
    static_assert(BN >= 16 && BN <= kBNMax && BN % 16 == 0, "MMA N with M = 128");
    constexpr int XB = BN * kBK * 2;                     // bytes of one X stage
    constexpr int kChunks = ((BN < 128 ? BN : 128) + 31) / 32;   // 32-column drains per epilogue warp
    // 16-byte ring slots per thread and stage: 8-bit kSliceK bytes; 4-bit kSliceK / 2
    // bytes; 3-bit one 12-byte group per slot (a 16-k slice copies its whole group)
    constexpr int SLOTS = EIGHT ? (kSliceK >= 16 ? kSliceK / 16 : 1) : (kSliceK == 64 ? 2 : 1);
    // code stages in flight per decode thread: as many as the free halves of the
    // table rows hold, at most 7
    constexpr int RING_FIT = (256 * 128) / (SLOTS * kCodeStageBytes);
    constexpr int RING = RING_FIT < 7 ? RING_FIT : 7;
    static_assert(RING * SLOTS * kCodeStageBytes <= 256 * 128, "code ring must fit in the table rows' free halves");
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    // Layout: pair table (code ring in its rows' free halves) | X stages | barriers
    const uint32_t sbase = smem_u32(smem_raw);
    const uint32_t xs0 = sbase + kTabRegion;
    const uint32_t bar0 = xs0 + kXStages * XB;
    const uint32_t layout_end = bar0 + 256;
    // the lookups address the table as an offset from kTabOff; refuse a launch
    // whose shared window differs or is too small for this layout
    if (sbase != kTabOff || layout_end > sbase + p.smem_bytes) {
        if (threadIdx.x == 0) {
            atomicExch(&p.ws->detail, (uint32_t)kWaitLayout);
            atomicExch(&p.ws->error, (uint32_t)LOGQ_ERR_TIMEOUT);
        }
        return;
    }
    // code-ring slot j of ring stage g: 16 bytes in the free half of table row
    // g * 32 * SLOTS + j / 8 (decode thread d owns slots SLOTS * d .. +SLOTS-1)
    auto ring_slot = [&](int g, int j) -> uint32_t {
        return sbase + (uint32_t)(g * (SLOTS * kDecodeThreads / 8) + (j >> 3)) * kTabRow + 128u +
               ((uint32_t)(j & 7) << 4);
    };
    uint8_t* gen = smem_raw - sbase;                  // generic pointer = gen + shared address
    // barriers: xfull[X], xempty[X], wfull[W], wempty[W], accfull, accempty, drain,
    // then the tmem slot and the abort flag
    auto xfull = [&](int s) { return bar0 + 8u * s; };
    auto xempty = [&](int s) { return bar0 + 8u * (kXStages + s); };
    auto wfull = [&](int s) { return bar0 + 8u * (2 * kXStages + s); };
    auto wempty = [&](int s) { return bar0 + 8u * (2 * kXStages + kWStages + s); };
    constexpr int kB0 = 2 * kXStages + 2 * kWStages;
    const uint32_t accfull = bar0 + 8u * kB0;
    const uint32_t accempty = bar0 + 8u * (kB0 + 1);
    const uint32_t drainb = bar0 + 8u * (kB0 + 2);
    const uint32_t tmem_slot = bar0 + 8u * (kB0 + 3);
    static_assert(8 * (2 * kXStages + 2 * kWStages + 3) + 8 + 4 <= 256, "barrier block overflows");
    volatile int* abort_flag = reinterpret_cast<volatile int*>(gen + tmem_slot + 8);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // this CTA's matrix, and its place among that matrix's CTAs
    int m = 0;
#pragma unroll
    for (int i = 1; i < kMaxPrefillItems; ++i)
        if (i < p.nitems && (int)blockIdx.x >= p.item[i].cta_begin) m = i;
    const PrefillItem& item = p.item[m];
    const int cta = (int)blockIdx.x - item.cta_begin, ncta = item.ncta;
    const uint8_t* const codes = item.codes;
    const int64_t N = item.N;
    const int n_tiles_n = item.n_tiles_n;
    if (tid == 0) {
        for (int s = 0; s < kXStages; ++s) {
            mbar_init(xfull(s), 1);
            mbar_init(xempty(s), 1);
        }
        for (int s = 0; s < kWStages; ++s) {
            mbar_init(wfull(s), kDecodeWarps);
            mbar_init(wempty(s), 1);
        }
        mbar_init(accfull, 1);
        mbar_init(accempty, kEpiWarps);
        mbar_init(drainb, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&xmap) : "memory");
    }
    // pair table: entry e (two codes) = bf16x2 / f16x2 of their levels, one copy per lane
    {
        const int nent = (EIGHT || p.bits == 4) ? 256 : 64;
        for (int i = tid; i < nent * 8; i += kThreads) {
            const int e = i >> 3, part = i & 7;
            uint32_t v;
            if constexpr (EIGHT) {
                v = (uint32_t)item.lvl16[e] * 0x10001u;
            } else {
                const uint32_t lo = (p.bits == 4) ? (e & 15) : (e & 7);
                const uint32_t hi = (p.bits == 4) ? (e >> 4) : (e >> 3);
                v = (uint32_t)item.lvl16[lo] | ((uint32_t)item.lvl16[hi] << 16);
            }
            sts128(sbase + e * kTabRow + part * 16, v, v, v, v);
        }
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(tmem_slot),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *reinterpret_cast<volatile uint32_t*>(gen + tmem_slot);

    const int ksteps = p.K / kBK;
    const int ntiles = n_tiles_n * p.n_tiles_t * p.splits;
    // tile -> (weight-row tile, token tile, k range); the weight-row tile varies fastest
    auto tile_n = [&](int tile) { return tile % n_tiles_n; };
    auto tile_t = [&](int tile) { return (tile / n_tiles_n) % p.n_tiles_t; };
    auto tile_sp = [&](int tile) { return tile / (n_tiles_n * p.n_tiles_t); };
    auto k_begin = [&](int tile) { return tile_sp(tile) * p.ksplit; };
    auto k_end = [&](int tile) {
        const int e = (tile_sp(tile) + 1) * p.ksplit;
        return e < ksteps ? e : ksteps;
    };

    // the code rows of a tile are one contiguous block: ask L2 for it one
    // tile ahead so the decode warps' copies hit L2.  An epilogue warp issues
    // it: from the producer warp it delays the X loads behind it, and a CTA's
    // first tile is not prefetched, since its copies would only compete with
    // the decode warps' own loads of the same rows.
    auto prefetch_codes = [&](int tile) {
        if (tile >= ntiles) return;
        const int64_t n0 = (int64_t)tile_n(tile) * kBM;
        const int64_t rows = (N - n0) < kBM ? (N - n0) : kBM;
        const uint8_t* base = codes + n0 * p.row_bytes;
        if (p.splits == 1) {
            const int64_t bytes = rows * p.row_bytes;
            for (int64_t off = (int64_t)lane * 16384; off < bytes; off += 32 * 16384) {
                const int64_t nb = (bytes - off) < 16384 ? (bytes - off) : 16384;
                asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base + off), "r"((uint32_t)nb)
                             : "memory");
            }
            return;
        }
        // the tile's k range of each row, widened to 16-byte bounds inside the row
        // (row_bytes is a multiple of 16, and of the k-step count)
        const int64_t step_bytes = p.row_bytes / ksteps;
        const int64_t b0 = ((int64_t)k_begin(tile) * step_bytes) & ~(int64_t)15;
        int64_t b1 = ((int64_t)k_end(tile) * step_bytes + 15) & ~(int64_t)15;
        if (b1 > p.row_bytes) b1 = p.row_bytes;
        for (int64_t r = lane; r < rows; r += 32)
            asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base + r * p.row_bytes + b0),
                         "r"((uint32_t)(b1 - b0))
                         : "memory");
    };
    if (warp == 0) {
        // ---------------- TMA producer ----------------
        // The whole warp walks the loop (uniform operands); one elected lane issues.
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        uint32_t issued = 0, issued_par = 0;           // per stage: used at least once / parity of last load
        for (int tile = cta; tile < ntiles && ok; tile += ncta) {
            const int t0 = tile_t(tile) * BN;
            const int kb = k_begin(tile), ke = k_end(tile);
            for (int ks = kb; ks < ke; ++ks) {
                if (!warp_wait(xempty(stage), phase ^ 1u, abort_flag, p.ws, kWaitProducer)) {
                    ok = false;
                    break;
                }
                if (elect_one()) {
                    mbar_expect_tx(xfull(stage), XB);
                    tma_load_2d(xs0 + stage * XB, &xmap, ks * kBK, t0, xfull(stage));
                }
                __syncwarp();
                issued |= 1u << stage;
                issued_par = (issued_par & ~(1u << stage)) | (phase << stage);
                if (++stage == kXStages) { stage = 0; phase ^= 1u; }
            }
        }
        // every load this warp issued has landed before the CTA can leave
        if (lane == 0)
            for (int st = 0; st < kXStages; ++st)
                if (issued & (1u << st))
                    wait_bounded(xfull(st), (issued_par >> st) & 1u, abort_flag, p.ws, kWaitDrain, true);
        __syncwarp();
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        // The whole warp walks the loop, so descriptors and addresses stay
        // warp-uniform; one elected lane issues the MMAs and commits.
        int xs = 0, wsg = 0;
        uint32_t xph = 0, wph = 0;
        bool ok = true;
        int it = 0;
#ifdef LOGQ_TEST_WAIT_HOOK
        // Test builds only (never the shipped library): when the caller's
        // workspace holds kTestStallWord, the MMA warp first waits on the drain
        // barrier, which nothing completes before the teardown, so that wait
        // runs out of its bound and the abort path of every role runs.
        if (p.ws->reserved[0] == kTestStallWord)
            ok = warp_wait(drainb, 0, abort_flag, p.ws, kWaitMma);
#endif
        for (int tile = cta; tile < ntiles && ok; tile += ncta, ++it) {
            // one accumulator: the epilogue has read the previous tile's out of it
            if (!warp_wait(accempty, ((uint32_t)it & 1u) ^ 1u, abort_flag, p.ws, kWaitMma)) break;
            tc_fence_after();
            const uint32_t dcol = tmem_base;
            const int kb = k_begin(tile), ke = k_end(tile);
            for (int ks = kb; ks < ke; ++ks) {
                if (!warp_wait(xfull(xs), xph, abort_flag, p.ws, kWaitMma) ||
                    !warp_wait(wfull(wsg), wph, abort_flag, p.ws, kWaitMma)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t acol = tmem_base + kWCol0 + (uint32_t)wsg * kWStageCols;
                const uint64_t bdesc = smem_desc_sw128(xs0 + xs * XB);
                if (elect_one()) {
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk) {
                        // 16 k: 8 columns of A further on; 32 bytes (2 descriptor units)
                        // further inside B's swizzle atom
                        mma_f16_ta(dcol, acol + 8 * kk, bdesc + 2 * kk, p.idesc, (ks != kb) || kk != 0);
                    }
                    mma_commit(xempty(xs));
                    mma_commit(wempty(wsg));
                }
                __syncwarp();
                if (++xs == kXStages) { xs = 0; xph ^= 1u; }
                if (++wsg == kWStages) { wsg = 0; wph ^= 1u; }
            }
            if (ok) {
                if (elect_one()) mma_commit(accfull);
                __syncwarp();
            }
        }
    } else if (warp >= kEpi0 && warp < kDec0) {
        // ---------------- epilogue ----------------
        // Two warps per TMEM lane quarter, each owning 128 of the tile's 256 token
        // columns.  16-bit outputs are read out of tensor memory and rounded into
        // registers first, so the accumulator is handed back before the stores.
        const int quarter = warp & 3;                   // TMEM lanes 32*quarter .. +31
        const int ehalf = (warp - kEpi0) >> 2;          // token columns 128*ehalf .. +127
        const int row = quarter * 32 + lane;
        const uint32_t tq = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(ehalf * 128);
        int it = 0;
        // an epilogue warp of the second column half, idle in 16-token tiles
        const bool pf_warp = warp == kEpi0 + 4;
        for (int tile = cta; tile < ntiles; tile += ncta, ++it) {
            if (pf_warp) prefetch_codes(tile + ncta);
            if (!warp_wait(accfull, (uint32_t)it & 1u, abort_flag, p.ws, kWaitEpilogue)) break;
            tc_fence_after();
            const int64_t n = (int64_t)tile_n(tile) * kBM + row;
            const int tb0 = tile_t(tile) * BN + ehalf * 128;
            // tokens of this half that exist (may be <= 0: the tile is narrower, or past B)
            const int hcols = (BN - ehalf * 128) < 128 ? (BN - ehalf * 128) : 128;
            const int jmax = (p.B - tb0) < hcols ? (p.B - tb0) : hcols;
            if (hcols <= 0) {
                // no column of this tile in this half: only hand the accumulator back
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(accempty);
            } else if (p.splits > 1 || p.y_dtype == LOGQ_F32) {
                // fp32 out: Y itself, or this k range's partial sums
                float* yb = p.splits > 1 ? item.part + (int64_t)tile_sp(tile) * p.B * N : static_cast<float*>(item.Y);
#pragma unroll 1
                for (int c = 0; c < kChunks; ++c) {
                    uint32_t v[32];
                    tmem_ld32(tq + (uint32_t)(c * 32), v);
                    const int jm = jmax - 32 * c;
                    if (n < N && jm > 0) {
                        float* y = yb + (int64_t)(tb0 + 32 * c) * N + n;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < jm) y[(int64_t)j * N] = __uint_as_float(v[j]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(accempty);
            } else {
                const bool bf = p.y_dtype == LOGQ_BF16;
                uint32_t pk[64];                        // tokens 2j, 2j+1 rounded to 16 bits
#pragma unroll
                for (int c = 0; c < kChunks; ++c) {
                    uint32_t v[32];
                    tmem_ld32(tq + (uint32_t)(c * 32), v);
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const float a = __uint_as_float(v[2 * j]), b = __uint_as_float(v[2 * j + 1]);
                        if (bf) {
                            const __nv_bfloat162 h2 = __floats2bfloat162_rn(a, b);
                            pk[16 * c + j] = *reinterpret_cast<const uint32_t*>(&h2);
                        } else {
                            const __half2 h2 = __floats2half2_rn(a, b);
                            pk[16 * c + j] = *reinterpret_cast<const uint32_t*>(&h2);
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(accempty);
                if (n < N && jmax > 0) {
                    // lanes hold consecutive n: each store instruction writes one
                    // contiguous run of Y[t][n0 .. n0+31]
                    uint16_t* y = static_cast<uint16_t*>(item.Y) + (int64_t)tb0 * N + n;
                    if (jmax == 128) {
#pragma unroll
                        for (int j = 0; j < 64; ++j) {
                            y[(int64_t)(2 * j) * N] = (uint16_t)(pk[j] & 0xffffu);
                            y[(int64_t)(2 * j + 1) * N] = (uint16_t)(pk[j] >> 16);
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 64; ++j) {
                            if (2 * j < jmax) y[(int64_t)(2 * j) * N] = (uint16_t)(pk[j] & 0xffffu);
                            if (2 * j + 1 < jmax) y[(int64_t)(2 * j + 1) * N] = (uint16_t)(pk[j] >> 16);
                        }
                    }
                }
            }
        }
    } else {
        // ---------------- decode ----------------
        // tcgen05.st reaches only the warp's TMEM lane quarter (warp % 4), so the
        // weight row of a thread is its TMEM lane: row = 32 * (warp % 4) + lane.
        // The warps of a quarter split the stage's 64 k into kSlices slices.
        const int dw = warp - kDec0;                    // 0 .. kDecodeWarps-1
        const int d = dw * 32 + lane;                   // code-ring slot, 0 .. kDecodeThreads-1
        const int r = (warp & 3) * 32 + lane;           // weight row within the tile
        const int h = dw >> 2;                          // slice: k kSliceK*h .. +kSliceK-1 of the stage
        const uint32_t tw = tmem_base + ((uint32_t)((warp & 3) * 32) << 16) + kWCol0 + (uint32_t)(kSlicePairs * h);
        const uint32_t lane4 = 4u * (uint32_t)lane;
        // bytes of one row's codes per stage, and where this thread's slice (for 3-bit:
        // the 32-k group holding it) starts among them
        const int step_bytes = EIGHT ? 64 : (p.bits == 4) ? 32 : 24;
        const int slice_off = EIGHT ? kSliceK * h : (p.bits == 4) ? (kSliceK / 2) * h : 12 * ((kSliceK * h) / 32);
        int stage = 0;
        uint32_t phase = 0;
        int total = 0;                                  // stages this CTA decodes
        for (int t = cta; t < ntiles; t += ncta) total += k_end(t) - k_begin(t);
        // Cursor over (tile, k-step) advanced without divisions: one for the
        // copies issued ahead, one for the stage being decoded.
        struct Cursor {
            int tile, ks, ke;                           // k-step and end of the tile's k range
            bool valid;                                 // this thread's row exists
            const uint8_t* row;                         // its codes: slice, stage 0
        };
        auto set_tile = [&](Cursor& c, int tile) {
            c.tile = tile;
            c.ks = tile < ntiles ? k_begin(tile) : 0;
            c.ke = tile < ntiles ? k_end(tile) : 0;
            const int64_t n = (int64_t)tile_n(tile) * kBM + r;
            c.valid = tile < ntiles && n < N;
            c.row = codes + (c.valid ? n : 0) * p.row_bytes + slice_off;
        };
        auto step = [&](Cursor& c) {
            if (++c.ks >= c.ke) set_tile(c, c.tile + ncta);
        };
        Cursor ahead, cur;
        set_tile(ahead, cta);
        set_tile(cur, cta);
        auto issue = [&](int g) {
            if (g < total && ahead.valid) {
                const uint8_t* src = ahead.row + (int64_t)ahead.ks * step_bytes;
                const uint32_t dst = ring_slot(g % RING, SLOTS * d);
                if constexpr (EIGHT) {
#pragma unroll
                    for (int q = 0; q < SLOTS; ++q) cp_async_16(dst + 16 * q, src + 16 * q);
                } else if (p.bits == 4) {
                    if constexpr (kSliceK == 16) cp_async_8(dst, src);
                    else {
#pragma unroll
                        for (int q = 0; q < SLOTS; ++q) cp_async_16(dst + 16 * q, src + 16 * q);
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < SLOTS; ++q) {                // group q: 12 bytes into slot q
                        cp_async_4(dst + 16 * q, src + 12 * q);
                        cp_async_4(dst + 16 * q + 4, src + 12 * q + 4);
                        cp_async_4(dst + 16 * q + 8, src + 12 * q + 8);
                    }
                }
            }
            if (g < total) step(ahead);
            cp_async_commit();
        };
        // Resolve the codes of one stage (its slot in the ring) into the slice's pair values.
        auto resolve = [&](int slot, bool valid, uint32_t (&pr)[kSlicePairs]) {
            if constexpr (EIGHT) {
                // word i holds the codes of k = kSliceK h + 4i .. +3: pairs 2i and 2i + 1
                constexpr int NWD = kSliceK / 4;
                uint32_t cw8[NWD];
#pragma unroll
                for (int q = 0; q < NWD / 4; ++q) {
                    uint4 c0 = make_uint4(0, 0, 0, 0);
                    if (valid) c0 = lds128(ring_slot(slot, SLOTS * d) + 16 * q);
                    cw8[4 * q] = c0.x; cw8[4 * q + 1] = c0.y; cw8[4 * q + 2] = c0.z; cw8[4 * q + 3] = c0.w;
                }
#pragma unroll
                for (int i = 0; i < NWD; ++i) {
                    const uint32_t v0 = lds_tab(prmt(cw8[i], lane4, 0x7604u));
                    const uint32_t v1 = lds_tab(prmt(cw8[i], lane4, 0x7614u));
                    const uint32_t v2 = lds_tab(prmt(cw8[i], lane4, 0x7624u));
                    const uint32_t v3 = lds_tab(prmt(cw8[i], lane4, 0x7634u));
                    pr[2 * i] = prmt(v0, v1, 0x5410u);
                    pr[2 * i + 1] = prmt(v2, v3, 0x5410u);
                }
            } else {
                uint32_t cw[4 * SLOTS];
    #pragma unroll
                for (int q = 0; q < SLOTS; ++q) {
                    uint4 cv = make_uint4(0, 0, 0, 0);
                    if (valid) cv = lds128(ring_slot(slot, SLOTS * d) + 16 * q);
                    cw[4 * q] = cv.x; cw[4 * q + 1] = cv.y; cw[4 * q + 2] = cv.z; cw[4 * q + 3] = cv.w;
                }
                if (p.bits == 4) {
                    // word i holds k = kSliceK h + 8i .. +7
    #pragma unroll
                    for (int i = 0; i < kSliceK / 8; ++i) {
                        const uint32_t c = cw[i];
                        pr[4 * i + 0] = lds_tab(prmt(c, lane4, 0x7604u));
                        pr[4 * i + 1] = lds_tab(prmt(c, lane4, 0x7614u));
                        pr[4 * i + 2] = lds_tab(prmt(c, lane4, 0x7624u));
                        pr[4 * i + 3] = lds_tab(prmt(c, lane4, 0x7634u));
                    }
                } else {
                    // one 12-byte group of 32 k: pair q (k 2q, 2q + 1) is the 6-bit field q % 5
                    // of word q / 5 (q < 15); pair 15 takes the two top bits of each word
                    // group gi's words are cw[4 gi .. 4 gi + 2] (its ring slot)
                    auto pair_off = [&](int q, int gi = 0) -> uint32_t {
                        const uint32_t* g3 = cw + 4 * gi;
                        if (q == 15)
                            return ((g3[0] >> 22) & 0x0300u) | ((g3[1] >> 20) & 0x0c00u) | ((g3[2] >> 18) & 0x3000u) | lane4;
                        const int f = q % 5;
                        const uint32_t x = g3[q / 5];
                        const uint32_t field = f == 0 ? (x << 8) : f == 1 ? (x << 2) : f == 2 ? (x >> 4)
                                             : f == 3 ? (x >> 10) : (x >> 16);
                        return (field & 0x3f00u) | lane4;
                    };
                    if constexpr (kSliceK == 64) {
    #pragma unroll
                        for (int q = 0; q < 32; ++q) pr[q] = lds_tab(pair_off(q & 15, q >> 4));
                    } else if constexpr (kSliceK == 32) {
    #pragma unroll
                        for (int q = 0; q < 16; ++q) pr[q] = lds_tab(pair_off(q));
                    } else {
                        // this slice is half of the group: pairs 8 (h & 1) .. +7
                        if ((h & 1) == 0) {
    #pragma unroll
                            for (int q = 0; q < 8; ++q) pr[q] = lds_tab(pair_off(q));
                        } else {
    #pragma unroll
                            for (int q = 0; q < 8; ++q) pr[q] = lds_tab(pair_off(8 + q));
                        }
                    }
                }
            }
        };
        // Software pipeline: the pairs of stage g+1 are looked up while stage g
        // waits for its weight slot and is stored.
        for (int g = 0; g < RING - 1; ++g) issue(g);
        uint32_t pr_a[kSlicePairs], pr_b[kSlicePairs];
        int slot = 0;                                   // ring slot of stage g
        if (total > 0) {
            issue(RING - 1);
            cp_async_wait<RING - 1>();
            resolve(slot, cur.valid, pr_a);
            step(cur);
        }
        // One stage: look up the next stage's pairs into nxt, then store this
        // stage's (cur) once its weight slot is free.  Called with the two
        // buffers in alternating roles, so no pairs are copied.
        bool ok = true;
        auto stage_step = [&](int g, const uint32_t (&cur_pr)[kSlicePairs], uint32_t (&nxt_pr)[kSlicePairs]) {
            if (++slot == RING) slot = 0;
            if (g + 1 < total) {
                issue(g + RING);
                cp_async_wait<RING - 1>();
                resolve(slot, cur.valid, nxt_pr);
                step(cur);
            }
            if (!warp_wait(wempty(stage), phase ^ 1u, abort_flag, p.ws, kWaitDecode)) {
                ok = false;
                return;
            }
            tc_fence_after();
            // pair q holds k = kSliceK h + 2q (low half) and + 1: column kSlicePairs h + q of the stage
            tmem_st_pairs(tw + (uint32_t)stage * kWStageCols, cur_pr);
            tmem_wait_st();
            tc_fence_before();            // this warp's tensor-memory writes -> the MMA issuer
            __syncwarp();
            if (lane == 0) mbar_arrive(wfull(stage));
            if (++stage == kWStages) { stage = 0; phase ^= 1u; }
        };
        for (int g = 0; g < total && ok; g += 2) {
            stage_step(g, pr_a, pr_b);
            if (g + 1 >= total || !ok) break;
            stage_step(g + 1, pr_b, pr_a);
        }
        cp_async_wait<0>();
    }

    // teardown: every MMA this CTA issued has completed before TMEM is freed
    __syncthreads();
    if (warp == 1) {
        if (elect_one()) {
            mma_commit(drainb);
            wait_bounded(drainb, 0, abort_flag, p.ws, kWaitDrain, true);
        }
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(kTmemCols)
                     : "memory");
    }
}

// ------------------------------------------------------------------ host ---

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

uint32_t make_idesc(bool f16_inputs, int bn)
{
    uint32_t d = 0;
    d |= 1u << 4;                                   // D format: fp32
    const uint32_t ab = f16_inputs ? 0u : 1u;       // A/B format: fp16 = 0, bf16 = 1
    d |= ab << 7;
    d |= ab << 10;
    // bits 15, 16: A and B K-major (0)
    d |= (uint32_t)(bn >> 3) << 17;                 // N / 8
    d |= (uint32_t)(kBM >> 4) << 24;                // M / 16
    return d;
}

// Dynamic shared memory of the layout: table rows, X stages, barriers.
constexpr uint32_t smem_bytes_for(int bn) { return kTabRegion + kXStages * (uint32_t)bn * kBK * 2 + 256; }

// Outputs of a split launch: per matrix its partial sums [splits][count] and Y[count].
struct SumArgs {
    const float* part[kMaxPrefillItems];
    void* Y[kMaxPrefillItems];
    int64_t count[kMaxPrefillItems];        // B * N
    int n;
};

// Fixed-order sum of the k ranges' fp32 partial sums: Y[i] = sum_s part[s][i]
// (s = 0, 1, ...), rounded to Y's dtype, over the matrices of the launch in turn.
__global__ void __launch_bounds__(256) splitk_sum_kernel(const __grid_constant__ SumArgs a, int splits, int64_t total,
                                                         int y_dtype)
{
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
        int m = 0;
        int64_t i = g;
        while (m + 1 < a.n && i >= a.count[m]) i -= a.count[m++];
        const float* part = a.part[m];
        const int64_t count = a.count[m];
        float v = part[i];
        for (int sp = 1; sp < splits; ++sp) v += part[(int64_t)sp * count + i];
        if (y_dtype == LOGQ_F32) static_cast<float*>(a.Y[m])[i] = v;
        else if (y_dtype == LOGQ_BF16) static_cast<__nv_bfloat16*>(a.Y[m])[i] = __float2bfloat16_rn(v);
        else static_cast<__half*>(a.Y[m])[i] = __float2half_rn(v);
    }
}

template <bool EIGHT, int BN>
cudaError_t launch(PrefillParams& p, const CUtensorMap& xmap, int grid, cudaStream_t s)
{
    constexpr uint32_t kSmemBytes = smem_bytes_for(BN);
    static uint32_t configured[64] = {0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev]) {
        int reserved = 0, optin = 0;
        if ((e = cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev)) != cudaSuccess) return e;
        if ((e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess) return e;
        const uint32_t bytes = kSmemBytes;
        if (reserved != (int)kTabOff || bytes > (uint32_t)optin) return cudaErrorNotSupported;
        e = cudaFuncSetAttribute(prefill_kernel<EIGHT, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
        if (e != cudaSuccess) return e;
        configured[dev] = bytes;
    }
    p.smem_bytes = configured[dev];
    prefill_kernel<EIGHT, BN><<<grid, kThreads, configured[dev], s>>>(p, xmap);
    return cudaGetLastError();
}

}  // namespace

PrefillPlan prefill_plan(int64_t B, const int64_t* N, int count, int64_t K, size_t part_bytes_avail)
{
    PrefillPlan pl;
    memset(&pl, 0, sizeof pl);
    pl.bn = B <= 16 ? 16 : kBNMax;
    const int sms = sm_count() > 0 ? sm_count() : 148;
    const int64_t ttiles = (B + pl.bn - 1) / pl.bn;
    int64_t tiles[kMaxPrefillItems], sum_n = 0;
    for (int i = 0; i < count; ++i) {
        tiles[i] = ((N[i] + kBM - 1) / kBM) * ttiles;
        sum_n += N[i];
    }
    const int64_t ksteps = K / kBK;
    // CTAs per matrix for `splits` k ranges per tile: one each, a share of the
    // rest of the grid in proportion to the matrix's work units, then each CTA
    // left over to the matrix whose CTAs take the most rounds (the grid never
    // exceeds the SMs).  Returns those rounds.
    auto share = [&](int64_t splits, int* ncta) -> int64_t {
        int64_t units[kMaxPrefillItems], total = 0;
        for (int i = 0; i < count; ++i) total += (units[i] = tiles[i] * splits);
        const int64_t grid = total < sms ? total : sms;
        int64_t used = 0;
        for (int i = 0; i < count; ++i) {
            int64_t c = 1 + (grid - count) * units[i] / total;
            c = c > units[i] ? units[i] : c;
            ncta[i] = (int)c;
            used += c;
        }
        auto rounds = [&](int i) { return (units[i] + ncta[i] - 1) / ncta[i]; };
        while (used < grid) {
            int best = -1;
            for (int i = 0; i < count; ++i) {
                if (ncta[i] >= units[i]) continue;
                if (best < 0 || rounds(i) > rounds(best) ||
                    (rounds(i) == rounds(best) && units[i] * ncta[best] > units[best] * ncta[i]))
                    best = i;
            }
            if (best < 0) break;
            ++ncta[best];
            ++used;
        }
        int64_t r = 0;
        for (int i = 0; i < count; ++i) r = rounds(i) > r ? rounds(i) : r;
        return r;
    };
    // Cost in k-step times (~0.5 us each on the GB300, for either tile width:
    // the roles' hand-offs and the decode threads' code copies, more than the
    // MMAs, set a stage's time): persistent CTAs take tiles in rounds,
    // a tile of ks k-steps costing ks + 6 (pipeline fill, and the MMA waiting
    // for the epilogue to drain the single accumulator).  A split adds the sum
    // kernel (~6) and the partial sums' HBM traffic, written once and read once
    // (8 bytes per output and range, at ~6 TB/s).  Each range keeps at least 8
    // k-steps and the partials fit the caller's workspace.  (Fitted to launches
    // of the Llama-3.1-8B shapes at batches 8-64 and 2048 tokens.)
    int ncta[kMaxPrefillItems];
    auto cost = [&](int64_t splits, int64_t ksplit) {
        double c = (double)share(splits, ncta) * (double)(ksplit + 6);
        if (splits > 1) c += 6.0 + (double)splits * (double)B * (double)sum_n * 8.0 / 3.0e6;
        return c;
    };
    pl.splits = 1;
    pl.ksplit = (int)ksteps;
    double best = cost(1, ksteps);
    for (int64_t sp = 2; sp <= 32 && ksteps / sp >= 8; ++sp) {
        const int64_t ksplit = (ksteps + sp - 1) / sp;
        const int64_t real = (ksteps + ksplit - 1) / ksplit;       // ranges actually used
        const size_t need = (size_t)real * (size_t)B * (size_t)sum_n * 4;
        if (need > part_bytes_avail) break;
        const double c = cost(real, ksplit);
        if (c < best) {
            best = c;
            pl.splits = (int)real;
            pl.ksplit = (int)ksplit;
        }
    }
    share(pl.splits, pl.ncta);
    pl.part_bytes = pl.splits > 1 ? (size_t)pl.splits * (size_t)B * (size_t)sum_n * 4 : 0;
    pl.est_us = 0.5 * best + 3.0;
    return pl;
}

PrefillPlan prefill_plan(int64_t B, int64_t N, int64_t K, size_t part_bytes_avail)
{
    return prefill_plan(B, &N, 1, K, part_bytes_avail);
}

namespace {

// One launch over `count` matrices that share X (and the split k ranges'
// sum kernel where the plan splits them).
cudaError_t launch_items(const GroupItem* gi, int count, const void* X, int x_f16, int64_t B, int64_t K, int bits,
                         int y_dtype, Workspace* ws, size_t ws_bytes, cudaStream_t s)
{
    auto encode = encode_fn();
    if (!encode) return cudaErrorNotSupported;
    int64_t Ns[kMaxPrefillItems];
    for (int i = 0; i < count; ++i) Ns[i] = gi[i].N;
    const size_t avail = ws_bytes > kWorkspaceBytes ? ws_bytes - kWorkspaceBytes : 0;
    const PrefillPlan pl = prefill_plan(B, Ns, count, K, avail);
    CUtensorMap xmap;
    memset(&xmap, 0, sizeof xmap);
    const cuuint64_t gdim[2] = {(cuuint64_t)K, (cuuint64_t)B};
    const cuuint64_t gstride[1] = {(cuuint64_t)K * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)pl.bn};
    const cuuint32_t estride[2] = {1, 1};
    CUresult r = encode(&xmap, x_f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(X), gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;

    PrefillParams p;
    memset(&p, 0, sizeof p);
    p.nitems = count;
    p.ws = ws;
    p.K = (int32_t)K;
    p.B = (int32_t)B;
    p.bits = bits;
    p.row_bytes = (bits == 8) ? K : (bits == 4) ? K / 2 : K / 32 * 12;
    p.y_dtype = y_dtype;
    p.n_tiles_t = (int32_t)((B + pl.bn - 1) / pl.bn);
    p.splits = pl.splits;
    p.ksplit = pl.ksplit;
    p.idesc = make_idesc(x_f16 != 0, pl.bn);
    // partial sums of matrix i after those of matrices 0 .. i-1
    float* part = pl.splits > 1 ? reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(ws) + kWorkspaceBytes) : nullptr;
    SumArgs sa;
    memset(&sa, 0, sizeof sa);
    sa.n = count;
    int grid = 0;
    int64_t total = 0;
    for (int i = 0; i < count; ++i) {
        PrefillItem& it = p.item[i];
        it.codes = gi[i].codes;
        it.Y = gi[i].Y;
        it.N = gi[i].N;
        it.n_tiles_n = (int32_t)((gi[i].N + kBM - 1) / kBM);
        it.cta_begin = grid;
        it.ncta = pl.ncta[i];
        it.part = part;
        for (int c = 0; c < (1 << bits); ++c) it.lvl16[c] = gi[i].lvl16[c];
        grid += pl.ncta[i];
        sa.part[i] = part;
        sa.Y[i] = gi[i].Y;
        sa.count[i] = B * gi[i].N;
        total += B * gi[i].N;
        if (part) part += (int64_t)pl.splits * B * gi[i].N;
    }

    cudaError_t e;
    if (pl.bn == 16)
        e = bits == 8 ? launch<true, 16>(p, xmap, grid, s) : launch<false, 16>(p, xmap, grid, s);
    else
        e = bits == 8 ? launch<true, kBNMax>(p, xmap, grid, s) : launch<false, kBNMax>(p, xmap, grid, s);
    if (e != cudaSuccess || pl.splits == 1) return e;
    const int sms = sm_count() > 0 ? sm_count() : 148;
    int64_t blocks = (total + 255) / 256;
    if (blocks > (int64_t)sms * 8) blocks = (int64_t)sms * 8;
    splitk_sum_kernel<<<(int)blocks, 256, 0, s>>>(sa, pl.splits, total, y_dtype);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_prefill(const LinearArgs& a, cudaStream_t s)
{
    GroupItem gi;
    memset(&gi, 0, sizeof gi);
    gi.codes = a.codes;
    gi.Y = a.Y;
    gi.N = a.N;
    for (int c = 0; c < (1 << a.bits); ++c) gi.lvl16[c] = a.lvl16[c];
    return launch_items(&gi, 1, a.X, a.x_f16, a.B, a.K, a.bits, a.y_dtype, a.ws, a.ws_bytes, s);
}

cudaError_t launch_prefill_group(const GroupArgs& g, size_t ws_bytes, cudaStream_t s)
{
    if (g.count < 1 || g.count > kMaxPrefillItems) return cudaErrorInvalidValue;
    return launch_items(g.item, g.count, g.X, g.x_f16, g.B, g.K, g.bits, g.y_dtype, g.ws, ws_bytes, s);
}

}  // namespace logq
