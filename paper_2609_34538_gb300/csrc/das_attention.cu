// das_attention.cu -- depth-asynchronous attention (Eqs. 2-3, Sec. 3.2) and
// the full-depth verify attention (Sec. 3.4) on the 5th-generation tensor
// cores of sm_103a (tcgen05, accumulators in tensor memory).
//
// Work decomposition: every (sequence, kv head) pair owns ceil(P/64) prefix
// tiles plus one block tile; all pairs' tiles form one list of N tiles, and
// CTA c of a persistent grid of C CTAs (one per SM) takes the c-th of C
// equal ranges of that list (block tiles weighted for their extra cost, see
// kBlockWeight), cut into segments at pair boundaries.  A segment that covers
// its pair writes the output.  The others write a partial (O / l and the
// log-sum-exp of their keys) to the workspace, and merge_kernel, launched
// right after as a programmatic dependent, combines each split pair's
// partials by log-sum-exp (8, 4 or 2 segments' loads in flight, chosen per
// launch).
//
// One CTA = four softmax warps + one TMA warp + two MMA warps (+ four
// conversion warps when prefix keys or values are stored as e4m3).
//   producer (warp 4): TMA loads of 64-key K and V tiles kStages ahead into a
//     ring of shared-memory stages, and of each segment's query rows (the
//     pair's G * max_block rows, ordered i * G + g, which is the order of a
//     {64, G, max_block} box).
//   P V issuer (warp 5) and S issuer (warp 6), one elected lane each, each
//   blocking on its own in-order barriers:
//       S = Q K^T    tcgen05.mma M=64 N=64 K=D   -> S buffer (k % 4) in TMEM
//                    (e4m3 keys at D = 128: two e4m3 passes over the query
//                    rows split exactly into hi + lo, see split_q)
//       O += P V     tcgen05.mma M=64 N=D K=64   -> O in TMEM
//       l += P 1     tcgen05.mma M=64 N=8 K=64   -> the rounded row sums
//     S of tile k is issued once its K has landed (or been widened) and the
//     softmax warps have read S buffer k % 4, so the tensor core runs up to
//     four tiles ahead of the softmax.  A stage is refilled once the P V that
//     read it has completed.
//   softmax warps: an M=64 MMA puts row r in TMEM lane 32 (r / 16) + r % 16, so
//     warp w owns rows 16w..16w+15 and two threads share a row (one per half
//     of the 64 keys).  They load the row's scores (and free the S buffer),
//     mask and scale them (base 2), keep a reference max m that only moves
//     when a score exceeds it by more than 2^8 (then O and l are rescaled in
//     TMEM), write P = 2^(s - m) as bf16 into a 128-byte-swizzled [64 rows]
//     [64 keys] buffer (the K-major A operand of P V) and accumulate the row
//     sum of the fp32 weights (for the lse).  The sum of the weights as
//     rounded to bf16 (for the normalisation, so that the output is a convex
//     combination of the values with exactly the weights the tensor core
//     used) is the tensor core's, P times a ones column.  At the end of a
//     segment they read the O rows and that sum from TMEM and write O / l and
//     the lse (or the partial).
// Pairs of at most 16 (32) query rows (decode-shaped calls; D = 128, bf16
// values, keys bf16 or e4m3 with split-query scores) take the
// replicated-rows variant: the rows are loaded four (two) times, at
// MMA rows 0, 16, 32 and 48 (0 and 32), and the softmax warps of copy c take
// only that copy's quarter (half) of every tile's keys, 8 (16) scores a
// thread instead of 32.  The rest of each copy's P row stays zero, so P V and
// the row-sum MMA accumulate each copy's own keys; each copy is a softmax of
// its own (reference max, sums, O rows), and the copies are combined by
// log-sum-exp through shared memory at a segment end.
// The kernel is launched as a programmatic dependent of the previous kernel
// in the stream: barrier set-up, the tensor-memory allocation, the work plan
// (from lengths read before the wait, checked again after it) and an L2
// prefetch of the first tiles overlap the previous kernel's tail; nothing
// global is written, and nothing read is used unchecked, before
// griddepcontrol.wait.  Every wait is bounded (2 s); a time-out sets the
// status word and stops the CTA's waits.  Tensor memory (512 columns) is
// freed before the CTA exits.
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>

#include "das_internal.h"

namespace das {
namespace tc {
namespace {

constexpr uint32_t kFull = 0xffffffffu;
constexpr unsigned long long kWaitNs = 2000000000ull;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kSoftWarps = 4;
constexpr int kProducerWarp = kSoftWarps;     // TMA loads
constexpr int kMmaWarp = kSoftWarps + 1;      // tcgen05 MMAs of P V
constexpr int kSWarp = kSoftWarps + 2;        // tcgen05 MMAs of S
constexpr int kConvWarp0 = kSoftWarps + 3;    // e4m3 -> bf16 widening (e4m3 variants)
constexpr int kConvWarps = 4;
constexpr int kRows = 64;            // M of every MMA (query rows per pair)
constexpr int kSBufs = 4;            // S buffers in tensor memory
constexpr int kPrefetchTiles = 2;    // prefix tiles pulled into L2 before the dependency wait
constexpr int kLongRange = 80;       // ranges longer than this prefetch one tile (measured:
                                     // long / verify 0.45 us faster, decode and batched not)
constexpr int kTmemCols = 512;       // S buffers [0, 64 kSBufs), O [64 kSBufs, 64 kSBufs + D),
                                     // then 8 columns whose first is the rounded row sum
constexpr float kRescaleLog2 = 8.f;  // move the reference max only beyond 2^8

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ unsigned long long globaltimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait; false after 2 s or once another thread of the CTA gave up.
__device__ __noinline__ bool wait_slow(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                       int32_t *status) {
    const unsigned long long t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 63u) == 0) {
            if (*abort_flag) return false;
            if (globaltimer() - t0 > kWaitNs) {
                *abort_flag = 1;
                atomicOr(status, kStatusWaitTimeout);
                return false;
            }
        }
    }
}
__device__ __forceinline__ bool wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                     int32_t *status) {
#pragma unroll 1
    for (int i = 0; i < 8; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    return wait_slow(bar, parity, abort_flag, status);
}

// On the abort path only: wait (at most 20 ms, whatever the abort flag says)
// for a phase whose completion also means that the copies signalling it
// have landed, so that no bulk copy into shared memory outlives the CTA.
__device__ __noinline__ void drain_wait(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(bar, parity) && globaltimer() - t0 < 20000000ull) {
    }
}

__device__ __forceinline__ void tma_5d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int c0,
                                       int c1, int c2, int c3, int c4, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%3, %4, %5, %6, %7}], [%2], %8;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
        "r"(c4), "l"(policy)
        : "memory");
}
// L2 prefetch of one box (no shared memory, no barrier).
__device__ __forceinline__ void tma_prefetch_5d(const CUtensorMap *map, int c0, int c1, int c2,
                                                int c3, int c4) {
    asm volatile("cp.async.bulk.prefetch.tensor.5d.L2.global.tile [%0, {%1, %2, %3, %4, %5}];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4)
                 : "memory");
}
__device__ __forceinline__ void tma_prefetch_4d(const CUtensorMap *map, int c0, int c1, int c2,
                                                int c3) {
    asm volatile("cp.async.bulk.prefetch.tensor.4d.L2.global.tile [%0, {%1, %2, %3, %4}];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(c3)
                 : "memory");
}
__device__ __forceinline__ void tma_4d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int c0,
                                       int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

// ---- tcgen05 ----------------------------------------------------------------
// Shared-memory matrix descriptor: start, leading / stride byte offsets,
// descriptor version 1, layout 2 = 128-byte swizzle.
__device__ __forceinline__ uint64_t sdesc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((addr >> 4) & 0x3FFF) | (uint64_t)((lbo >> 4) & 0x3FFF) << 16 |
           (uint64_t)((sbo >> 4) & 0x3FFF) << 32 | (uint64_t)1 << 46 | (uint64_t)2 << 61;
}
// Instruction descriptor of kind::f16: bf16 A and B, fp32 D, majors, N, M.
__host__ __device__ constexpr uint32_t idesc(int M, int N, int a_mn_major, int b_mn_major) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn_major << 15) |
           ((uint32_t)b_mn_major << 16) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t id,
                                    uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(id), "r"(accumulate)
        : "memory");
}
// kind::f8f6f4 with e4m3 A and B (format code 0 for both), fp32 D, both K-major.
__host__ __device__ constexpr uint32_t idesc_e4m3(int M, int N) {
    return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t id,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(id), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}
__device__ __forceinline__ void fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// true on exactly one lane of the (converged) warp
__device__ __forceinline__ bool elect_one() {
    uint32_t pred;
    asm volatile(
        "{\n .reg .pred P;\n .reg .b32 R;\n elect.sync R|P, 0xffffffff;\n"
        " selp.u32 %0, 1, 0, P;\n}\n"
        : "=r"(pred));
    return pred != 0;
}
// 32 lanes x 32 consecutive 32-bit columns; thread t gets lane (base + t).
// The load and its wait form one statement, so no use of the registers can
// be scheduled before the data is there.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}
// 32 columns of S for the calling thread (16 lanes x 2 halves): thread t < 16
// of a warp gets TMEM lane t, columns [c, c + 32), thread t + 16 the same lane,
// [c + 32, c + 64).  With M = 64 a warp's rows sit in its first 16 lanes, so
// two threads share each row.
__device__ __forceinline__ void tmem_ld_half32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], "
        "32;\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}
// (Replicated rows) the calling thread's 8 scores: lane t < 16 of the warp
// reads TMEM lane t, columns [0, 8) from taddr, lane t + 16 the same lane,
// columns [8, 16).
__device__ __forceinline__ void tmem_ld_half8(uint32_t taddr, float (&v)[8]) {
    uint32_t r[8];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8], 8;\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = __uint_as_float(r[j]);
}
// (Replicated rows, two copies) the calling thread's 16 scores: lane t < 16
// reads TMEM lane t, columns [0, 16) from taddr, lane t + 16 the same lane,
// columns [16, 32).
__device__ __forceinline__ void tmem_ld_half16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15}, [%16], 16;\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]);
}
// The O row of the calling thread's half: with M = 64, thread t < 16 of a warp
// gets TMEM lane t, columns [64 g, 64 g + 32) for g < D / 64, and thread t + 16
// the same lane, columns [64 g + 32, 64 g + 64).  All loads are issued before
// the single wait, so the epilogue pays one TMEM round trip.
template <int D>
__device__ __forceinline__ void tmem_ld_orow(uint32_t taddr, float (&v)[D / 2]);
template <>
__device__ __forceinline__ void tmem_ld_orow<128>(uint32_t taddr, float (&v)[64]) {
    uint32_t r[64];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%64], 32;\n"
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,"
        "%27,%28,%29,%30,%31}, [%65], 32;\n"
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,"
        "%43,%44,%45,%46,%47}, [%66], 32;\n"
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,"
        "%59,%60,%61,%62,%63}, [%67], 32;\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]),
          "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]),
          "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]),
          "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]),
          "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]),
          "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(taddr), "r"(taddr + 16), "r"(taddr + 64), "r"(taddr + 80)
        : "memory");
#pragma unroll
    for (int j = 0; j < 64; ++j) v[j] = __uint_as_float(r[j]);
}
template <>
__device__ __forceinline__ void tmem_ld_orow<64>(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%32], 32;\n"
        "tcgen05.ld.sync.aligned.16x32bx2.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,"
        "%27,%28,%29,%30,%31}, [%33], 32;\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr), "r"(taddr + 16)
        : "memory");
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(
            taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
        "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
        "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
        "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
        "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
        "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Packed fp32 arithmetic (two independent IEEE operations per instruction,
// bit for bit the scalar results) and the three-input maximum.
__device__ __forceinline__ void fma2(float &d0, float &d1, float a0, float a1, float b0, float b1,
                                     float c0, float c1) {
    asm("{\n .reg .b64 a, b, c, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
        " mov.b64 c, {%6, %7};\n fma.rn.f32x2 d, a, b, c;\n mov.b64 {%0, %1}, d;\n}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ void add2(float &d0, float &d1, float a0, float a1, float b0, float b1) {
    asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
        " add.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
__device__ __forceinline__ void mul2(float &d0, float &d1, float a0, float a1, float b0, float b1) {
    asm("{\n .reg .b64 a, b, d;\n mov.b64 a, {%2, %3};\n mov.b64 b, {%4, %5};\n"
        " mul.rn.f32x2 d, a, b;\n mov.b64 {%0, %1}, d;\n}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// ---- tile list ----------------------------------------------------------------
__device__ __forceinline__ int clamp_prefix(const AttnParams &p, int b) {
    int v = p.prefix_len[b];
    return v < 0 ? 0 : (v > p.capacity ? p.capacity : v);
}
__device__ __forceinline__ int clamp_block(const AttnParams &p, int b) {
    int v = p.block_len[b];
    return v < 0 ? 0 : (v > p.max_block ? p.max_block : v);
}
__device__ __forceinline__ int tiles_of(int P) { return (P + kTileKeys - 1) / kTileKeys + 1; }

struct Walk {
    int b, h, t, nt, P, T;
};
__device__ __forceinline__ void walk_load_seq(const AttnParams &p, Walk &w) {
    if (w.b < p.B) {
        w.P = clamp_prefix(p, w.b);
        w.T = clamp_block(p, w.b);
        w.nt = tiles_of(w.P);
    }
}
__device__ __forceinline__ void walk_next(const AttnParams &p, Walk &w) {
    if (++w.t == w.nt) {
        w.t = 0;
        if (++w.h == p.Hkv) {
            w.h = 0;
            ++w.b;
            walk_load_seq(p, w);
        }
    }
}

// Extra weight of a pair's block tile when the list is split.  Ending one
// segment and starting the next (the mostly empty block tile holding a
// pipeline slot, the wait for the last P V, the partial write, the next
// queries) costs a CTA two to three tiles' time (a fit of per-CTA loop times
// on the batched workload: about 1.1 us per block tile plus 0.65 us per
// segment, against 0.72 us per tile), so a range that holds a block tile
// takes three tiles fewer while there is at least one CTA per pair; with
// more pairs than CTAs nearly every range holds one and the weight would
// only move work around (weights 1-4 and CTA-per-pair thresholds 1 and 4
// measured on the decode, long, batched and verify workloads; 3 against 2:
// long 86.9 -> 86.7 us, the others within 0.1 %).
constexpr int kBlockWeight = 3;
constexpr int kCtasPerPairForWeight = 1;

// The split of the tile list: tile x of pair q has weighted position
// x + beta q; CTA c takes the tiles whose weighted position lies in
// [c W / C, (c+1) W / C).  beta = kBlockWeight if there are at least
// kCtasPerPairForWeight CTAs per pair and W >= (2 + beta) C (which leaves no
// CTA empty: weighted positions are at most 1 + beta apart), else 0.
struct Split {
    long long N;  // tiles
    long long W;  // N + beta * pairs
    int beta;
};

// The split, given the total tile count.
__device__ __forceinline__ Split split_from_total(const AttnParams &p, long long total) {
    const long long pairs = (long long)p.B * p.Hkv;
    Split sp;
    sp.N = total;
    sp.beta = pairs * kCtasPerPairForWeight <= p.num_ctas &&
                      total + kBlockWeight * pairs >= (long long)(2 + kBlockWeight) * p.num_ctas
                  ? kBlockWeight
                  : 0;
    sp.W = total + sp.beta * pairs;
    return sp;
}

// Clamped length read from L2 (not kept in L1, so that a value read before
// the dependency wait can never be served stale to a later load).
__device__ __forceinline__ int len_cg(const int32_t *a, int b, int cap) {
    const int v = __ldcg(a + b);
    return v < 0 ? 0 : (v > cap ? cap : v);
}

// Tiles of one pair of sequence b (0 past the batch); at most 2^25, so sums
// over 32 sequences fit in 32 bits.
__device__ __forceinline__ int seq_tiles(const AttnParams &p, int b) {
    return b < p.B ? tiles_of(clamp_prefix(p, b)) : 0;
}

__device__ Split split_of(const AttnParams &p) {  // whole warp
    const int lane = threadIdx.x & 31;
    long long total = 0;
    for (int b0 = 0; b0 < p.B; b0 += 32)
        total += (long long)__reduce_add_sync(kFull, (unsigned)seq_tiles(p, b0 + lane)) * p.Hkv;
    return split_from_total(p, total);
}

// a / b for 0 <= a, 0 < b: a 32-bit division when both fit (the usual case;
// a 64-bit division is a long dependent instruction sequence).
__device__ __forceinline__ long long udiv(long long a, long long b) {
    if ((((unsigned long long)a | (unsigned long long)b) >> 32) == 0)
        return (long long)((uint32_t)a / (uint32_t)b);
    return a / b;
}

// The CTA whose weighted range holds weighted position q.
__device__ __forceinline__ int cta_of_w(long long q, const Split &sp, int C) {
    return (int)udiv((q + 1) * C - 1, sp.W);
}

// Range [lo, hi) of this CTA and the walk state of its first tile (a whole
// warp executes this).  One pass over the sequences: a 32-bit inclusive scan
// of the per-pair tile counts gives, for sequence b of a chunk, both the
// tiles and the weighted positions before it; the tiles at the weighted
// positions c W / C and (c+1) W / C are located in the same pass.
// P0 / T0: the clamped lengths of sequence `lane` (0 past the batch), given
// by the caller; with B <= 32 they are all the plan reads.
__device__ bool plan(const AttnParams &p, int P0, int T0, long long &lo, long long &hi, Walk &w) {
    const int lane = threadIdx.x & 31;
    const int nt0 = lane < p.B ? tiles_of(P0) : 0;
    const Split sp =
        p.B <= 32 ? split_from_total(p, (long long)__reduce_add_sync(kFull, (unsigned)nt0) * p.Hkv)
                  : split_of(p);
    const long long lw = udiv((long long)blockIdx.x * sp.W, p.num_ctas);
    const long long hw = udiv(((long long)blockIdx.x + 1) * sp.W, p.num_ctas);
    lo = hi = sp.N;
    bool have_lo = false;
    long long run_w = 0, run_t = 0;  // weighted positions / tiles before the chunk
    for (int b0 = 0; b0 < p.B; b0 += 32) {
        const int nt = b0 == 0 ? nt0 : seq_tiles(p, b0 + lane);
        int inc = nt;  // inclusive scan over the chunk
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const int u = __shfl_up_sync(kFull, inc, d);
            if (lane >= d) inc += u;
        }
        const int nseq = min(32, p.B - b0);
        // weighted position after this lane's sequence
        const long long after_w =
            run_w + ((long long)inc + (long long)sp.beta * min(lane + 1, nseq)) * p.Hkv;
        // tile x at weighted position q, q inside sequence f of this chunk
        auto locate = [&](long long q, int f, Walk *wk) {
            const int ntf = __shfl_sync(kFull, nt, f);
            const int excl = __shfl_sync(kFull, inc, f) - ntf;
            const long long seq_w = run_w + ((long long)excl + (long long)sp.beta * f) * p.Hkv;
            const long long seq_t = run_t + (long long)excl * p.Hkv;
            const long long off = q - seq_w;
            int h = (int)udiv(off, ntf + sp.beta);
            int t = (int)(off - (long long)h * (ntf + sp.beta));
            if (t >= ntf) {  // inside a block tile's extra weight: the next pair
                t = 0;
                ++h;
            }
            if (wk) {
                wk->b = b0 + f;
                wk->h = h;
                wk->t = t;
                if (b0 == 0) {  // lengths already in registers
                    wk->P = __shfl_sync(kFull, P0, f);
                    wk->T = __shfl_sync(kFull, T0, f);
                    wk->nt = tiles_of(wk->P);
                } else {
                    walk_load_seq(p, *wk);
                }
                if (wk->h == p.Hkv) {
                    wk->h = 0;
                    ++wk->b;
                    walk_load_seq(p, *wk);
                }
            }
            return seq_t + (long long)h * ntf + t;
        };
        if (!have_lo) {
            const unsigned m = __ballot_sync(kFull, after_w > lw);
            if (m) {
                lo = locate(lw, __ffs(m) - 1, &w);
                have_lo = true;
            }
        }
        if (have_lo) {
            const unsigned m = __ballot_sync(kFull, after_w > hw);
            if (m) {
                hi = locate(hw, __ffs(m) - 1, nullptr);
                break;
            }
        }
        run_w += ((long long)__shfl_sync(kFull, inc, 31) + (long long)sp.beta * nseq) * p.Hkv;
        run_t += (long long)__shfl_sync(kFull, inc, 31) * p.Hkv;
    }
    return lo < hi;
}

// Shared memory of one CTA.  Keys and values stored as e4m3 (the depths below
// R in a das_kv_cache_f8) land in the stage as 8-bit tiles [64 keys][D].
//   kQSplit (keys e4m3, values bf16, D = 128: Mature-V over a das_kv_cache_f8):
//     the key tile lands 128-byte swizzled and is read by the S MMAs as it is
//     (kind::f8f6f4).  The conversion warps split each segment's bf16 query
//     rows exactly into two e4m3 parts, 2^e q = hi + lo with one power of two
//     e per row (see split_q), and S = (hi + lo) K^T is two e4m3 products
//     accumulated in fp32, 2^e times the bf16 product.  The pair's block
//     tile (bf16 keys) has a bf16 key buffer of its own and bf16 MMAs.
//   otherwise: the conversion warps widen every e4m3 tile into bf16 tiles, in
//     the 128-byte-swizzled layout the MMAs read, held in a ring of kConvSlots
//     slots (tile j in slot j % kConvSlots) rather than one per stage: the
//     smaller stages then fit 6 (or 7) deep instead of 4, which is what keeps
//     more DRAM requests in flight per SM.  A pair's block tile is bf16: the
//     conversion warps load its e4m3-stored operands straight into the ring
//     slot, the producer the others into the stage.
template <int D, bool KF8, bool VF8, int NC = 1>
struct Layout {
    static constexpr bool REP = NC > 1;  // NC copies of the query rows (1, 2 or 4)
    static_assert(NC == 1 || NC == 2 || NC == 4, "copies: 1, 2 or 4");
    // bf16 keys, or e4m3 keys with the split-query scores; bf16 values; D = 128
    static_assert(!REP || (!VF8 && D == 128), "replicated rows: bf16 values, D = 128");
    static constexpr bool kQSplit = KF8 && !VF8 && D == 128;
    static constexpr bool kConv = KF8 || VF8;
    // (kQSplit: 4 stages of 24 KB measured faster than 5, e4m3 long 82.0 -> 81.5 us)
    static constexpr int kStages = kQSplit ? 4 : (KF8 && VF8) ? 7 : kConv ? 6 : 4;
    static constexpr int kConvSlots = 2;
    static constexpr int kThreads = (kSoftWarps + 3 + (kConv ? kConvWarps : 0)) * 32;
    static constexpr int kPanels = D / 64;
    static constexpr int kTileBytes = kTileKeys * D * 2;  // a bf16 K or V tile
    static constexpr int kTile8Bytes = kTileKeys * D;     // an e4m3 tile
    static constexpr int kKBytes = KF8 ? kTile8Bytes : kTileBytes;  // K part of a stage
    static constexpr int kVBytes = VF8 ? kTile8Bytes : kTileBytes;  // V part of a stage
    static constexpr int kStageBytes = kKBytes + kVBytes;
    static constexpr int kConvBytes =
        kQSplit ? 0 : (KF8 ? kTileBytes : 0) + (VF8 ? kTileBytes : 0);
    static constexpr int kQBytes = kPanels * kRows * 128;  // one query buffer
    static constexpr int kQ8Bytes = kRows * 128;           // one e4m3 query part (D = 128)
    static constexpr int kPBytes = kRows * kTileKeys * 2;  // one P buffer
    static constexpr int kStagesOff = 0;
    static constexpr int kConvOff = kStages * kStageBytes;  // the ring of widened tiles, or
    // (kQSplit) the block tile's bf16 keys, then hi / lo of both query buffers
    static constexpr int kBlkKOff = kConvOff;
    static constexpr int kQ8Off = kConvOff + kTileBytes;
    static constexpr int kExtraBytes =
        kQSplit ? kTileBytes + 4 * kQ8Bytes : kConvSlots * kConvBytes;
    static constexpr int kQOff = kConvOff + kExtraBytes;
    static constexpr int kPOff = kQOff + 2 * kQBytes;
    // the B operand of the row-sum MMA: [8][64] bf16, row 0 ones, 128-byte swizzled
    static constexpr int kOnesOff = kPOff + 2 * kPBytes;
    static constexpr int kBarOff = kOnesOff + 1024;
    // barriers: full[kStages], empty[kStages], qfull[2], qempty[2],
    // sready[kSBufs], sfree[kSBufs], pready[2], pvdone[2], drain[2],
    // cready[kConvSlots], kfree[kConvSlots], vfree[kConvSlots], qsplit[2], bkfree
    static constexpr int kNumBars = 2 * kStages + 10 + 2 * kSBufs + 3 * kConvSlots + 3;
    static constexpr int kMiscOff = kBarOff + kNumBars * 8;
    static constexpr int kLenOff = kMiscOff + 16;  // lengths read before the dependency wait
    static constexpr int kQeOff = kLenOff + 64 * 4;  // (kQSplit) e of each row, per query buffer
    // (REP) the segment end's exchange, then (m, l, rounded l) of every MMA
    // row [kRows][4]; rows are padded by 16 bytes so that consecutive rows
    // start in different bank groups.  Compacted (e4m3 keys, whose stages
    // leave too little shared memory for whole rows): a softmax thread holds
    // D / 2 values of its copy's O row, in NC groups of D / 2 / NC; each
    // group is combined by the thread of the copy with its index, so a thread
    // stores only the NC - 1 groups other copies combine: [2 halves][kRows]
    // [kXchStride] floats.
    // With bf16 keys there is room for the whole rows: every copy's O row
    // [kRows][kXchStride] (measured faster for bf16: decode 17.43 -> 17.12 us).
    static constexpr bool kCompactXch = KF8;
    static constexpr int kXchStride =
        !REP ? 0 : kCompactXch ? (NC - 1) * (D / 2 / NC) + 4 : D + 4;
    static constexpr int kXchOff = (kQeOff + (kQSplit ? 2 * kRows * 4 : 0) + 15) & ~15;
    static constexpr int kXchBytes =
        !REP ? 0
             : ((kCompactXch ? 2 * kRows * kXchStride : kRows * kXchStride) + kRows * 4) * 4;
    static constexpr int kBytes = kXchOff + kXchBytes + 1024;  // + alignment slack
    static_assert(kStageBytes % 1024 == 0 && kKBytes % 1024 == 0 && kConvBytes % 1024 == 0,
                  "swizzled tiles need 1024-byte alignment");
    static_assert(kBytes <= 232448, "shared memory per CTA");
};

// K-major 128B-swizzled address of bf16 element (row, col) of a [64][64] panel
__device__ __forceinline__ uint32_t p_chunk_addr(uint32_t base, int row, int chunk) {
    return base + row * 128 + ((chunk ^ (row & 7)) << 4);
}

// Two e4m3 codes (the low and high byte of a) -> bf16x2 (low, high half):
// the hardware conversion to f16x2 (exact: every e4m3 value, NaN included, is
// an f16 value), each half widened to f32 and the pair rounded to bf16x2
// (exact again: an e4m3 value has at most 4 significant bits).
__device__ __forceinline__ uint32_t e4m3x2_to_bf16x2(uint32_t a) {
    uint32_t h;
    asm("{\n .reg .b16 t;\n cvt.u16.u32 t, %1;\n cvt.rn.f16x2.e4m3x2 %0, t;\n}\n"
        : "=r"(h)
        : "r"(a));
    float f0, f1;
    asm("{\n .reg .b16 l, u;\n mov.b32 {l, u}, %2;\n cvt.f32.f16 %0, l;\n cvt.f32.f16 %1, u;\n}\n"
        : "=f"(f0), "=f"(f1)
        : "r"(h));
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(f1), "f"(f0));
    return r;
}

// Widen an e4m3 tile [64 keys][D] (row-major, as the 8-bit TMA box lands)
// into the bf16 tile the MMAs read: D / 64 panels of [64 keys][128 bytes],
// 16-byte chunk j of key r at (j ^ (r % 8)) * 16 (128-byte swizzle).  The 128
// conversion threads (ct = 0..127) each take 16-element chunks.
template <int D>
__device__ __forceinline__ void widen_tile(uint32_t src, uint32_t dst, int ct) {
    constexpr int kChunks = kTileKeys * D / 16;
#pragma unroll
    for (int i = 0; i < kChunks / (kConvWarps * 32); ++i) {
        const int c = ct + i * kConvWarps * 32;
        // Chunk c: 16 elements jj of a 64-column panel of a key.  The 8 lanes
        // of a quarter warp (one shared-memory wavefront of 16-byte accesses)
        // take two keys of opposite parity, so their loads (rows of D bytes)
        // and their swizzled stores each touch 8 distinct 16-byte bank groups.
        const int jj = c & 3;
        const int pnl = D == 128 ? (c >> 2) & 1 : 0;
        const int key = D == 128 ? ((c >> 4) << 1) + (pnl ^ ((c >> 3) & 1)) : c >> 2;
        const int d0 = pnl * 64 + jj * 16;
        uint32_t w0, w1, w2, w3;
        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
                     : "r"(src + key * D + d0));
        const uint32_t row = dst + (d0 / 64) * 8192 + key * 128;
        const int j = (d0 % 64) / 8;  // the first of two 16-byte bf16 chunks
        // bytes 0,1 / 2,3 of each word into the 16-bit halves of a register
        auto lo = [](uint32_t w) { return w & 0xFFFFu; };
        auto hi = [](uint32_t w) { return w >> 16; };
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                         row + ((j ^ (key & 7)) << 4)),
                     "r"(e4m3x2_to_bf16x2(lo(w0))), "r"(e4m3x2_to_bf16x2(hi(w0))),
                     "r"(e4m3x2_to_bf16x2(lo(w1))), "r"(e4m3x2_to_bf16x2(hi(w1)))
                     : "memory");
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                         row + (((j + 1) ^ (key & 7)) << 4)),
                     "r"(e4m3x2_to_bf16x2(lo(w2))), "r"(e4m3x2_to_bf16x2(hi(w2))),
                     "r"(e4m3x2_to_bf16x2(lo(w3))), "r"(e4m3x2_to_bf16x2(hi(w3)))
                     : "memory");
    }
}

// Exact split of the query rows for e4m3 keys (D = 128).  Row r of the bf16
// query buffer q (two 128-byte-swizzled panels of [64 rows][64 dims]) becomes
// two e4m3 rows hi, lo (128-byte swizzled [64 rows][128 dims]) with
//   2^e q = hi + lo,  e = 7 - floor(log2 max_d |q_d|)  (clamped to +-120),
// so that the row's largest element scales into [128, 256).  hi is 2^e q
// rounded to e4m3 (4 significant bits) and lo the rounded remainder: a bf16
// value has 8 significant bits, so the remainder fits e4m3 exactly unless it
// falls below e4m3's smallest subnormal (2^-9), i.e. for elements below about
// 2^-9 of the row's largest.  Thread ct of the 128 conversion threads takes
// row ct / 2, dims [64 (ct % 2), +64); e is written to qexp[row].  A row of
// zeros gives e = 0; the query must be finite.
__device__ __forceinline__ void split_q(uint32_t q, uint32_t hi, uint32_t lo, int *qexp, int ct) {
    const int row = ct >> 1, half = ct & 1;
    uint32_t w[32];
#pragma unroll
    for (int c = 0; c < 8; ++c)
        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(w[4 * c]), "=r"(w[4 * c + 1]), "=r"(w[4 * c + 2]), "=r"(w[4 * c + 3])
                     : "r"(q + half * (kRows * 128) + row * 128 + ((c ^ (row & 7)) << 4)));
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        mx = fmaxf(mx, fmaxf(fabsf(__uint_as_float(w[i] << 16)),
                             fabsf(__uint_as_float(w[i] & 0xffff0000u))));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    int e = 0;
    if (mx > 0.f && mx <= 3.4e38f) {
        e = 7 - ((int)((__float_as_uint(mx) >> 23) & 0xffu) - 127);
        e = e < -120 ? -120 : (e > 120 ? 120 : e);
    }
    const float sc = __uint_as_float((uint32_t)(127 + e) << 23);
    // word i holds dims 2i (low half) and 2i + 1 of the thread's 64
    uint32_t h[16], l[16];
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const float xa = __uint_as_float(w[i] << 16) * sc;
        const float xb = __uint_as_float(w[i] & 0xffff0000u) * sc;
        uint32_t h2, f2, l2;
        asm("{\n .reg .b16 t;\n cvt.rn.satfinite.e4m3x2.f32 t, %1, %2;\n cvt.u32.u16 %0, t;\n}"
            : "=r"(h2)
            : "f"(xb), "f"(xa));
        asm("{\n .reg .b16 t;\n cvt.u16.u32 t, %1;\n cvt.rn.f16x2.e4m3x2 %0, t;\n}"
            : "=r"(f2)
            : "r"(h2));
        float ha, hb;
        asm("{\n .reg .b16 a, b;\n mov.b32 {a, b}, %2;\n cvt.f32.f16 %0, a;\n cvt.f32.f16 %1, b;\n}"
            : "=f"(ha), "=f"(hb)
            : "r"(f2));
        asm("{\n .reg .b16 t;\n cvt.rn.satfinite.e4m3x2.f32 t, %1, %2;\n cvt.u32.u16 %0, t;\n}"
            : "=r"(l2)
            : "f"(xb - hb), "f"(xa - ha));
        if (i & 1) {
            h[i >> 1] |= h2 << 16;
            l[i >> 1] |= l2 << 16;
        } else {
            h[i >> 1] = h2;
            l[i >> 1] = l2;
        }
    }
    // 16-byte chunk c of the 128-byte e4m3 row holds dims 16 c .. 16 c + 15:
    // this thread's are chunks 4 half .. 4 half + 3
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        const uint32_t off = row * 128 + (((4 * half + m) ^ (row & 7)) << 4);
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(hi + off), "r"(h[4 * m]),
                     "r"(h[4 * m + 1]), "r"(h[4 * m + 2]), "r"(h[4 * m + 3])
                     : "memory");
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(lo + off), "r"(l[4 * m]),
                     "r"(l[4 * m + 1]), "r"(l[4 * m + 2]), "r"(l[4 * m + 3])
                     : "memory");
    }
    if (half == 0) qexp[row] = e;
}

// Registers a thread of the query-split variant may use: 144 x 352 threads
// leave room for one merge CTA (128 threads x 116) beside the attention CTA,
// so the merge kernel is resident before the attention grid ends (measured:
// the e4m3 long call 89.9 -> 89.0 us against 165 registers, no spills).
template <int D, bool KF8, bool VF8>
constexpr int kRegCap = Layout<D, KF8, VF8>::kQSplit ? 144 : 255;

// KF8 / VF8: prefix keys / values are e4m3 (tm_k / tm_v are 8-bit maps).
// NC > 1 (D = 128, bf16 values, at most 64 / NC query rows per pair):
// replicated rows.  The pair's rows are loaded NC times, copy c at MMA rows [c 64 / NC,
// (c + 1) 64 / NC), so that the softmax warps of copy c take only keys
// [c 64 / NC, (c + 1) 64 / NC) of each tile (32 / NC a thread instead of 32).
// The other keys of their P rows stay zero (the P buffers are cleared once),
// so P V accumulates each copy's own keys, and each copy keeps its own
// reference max, sums and O rows; at a segment end the copies are combined
// by log-sum-exp through shared memory.
template <int D, bool KF8, bool VF8, int NC>
__global__ void __launch_bounds__(Layout<D, KF8, VF8, NC>::kThreads, 1)
    __maxnreg__((kRegCap<D, KF8, VF8>)) attn_kernel(const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v,
                   const __grid_constant__ CUtensorMap tm_kb,
                   const __grid_constant__ CUtensorMap tm_vb,
                   const __grid_constant__ CUtensorMap tm_q, const AttnParams p) {
    using Lt = Layout<D, KF8, VF8, NC>;
    constexpr bool REP = Lt::REP;
    constexpr int kStages = Lt::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(sm);
    const uint32_t bars = sbase + Lt::kBarOff;
    const uint32_t b_full = bars, b_empty = bars + 8 * kStages, b_qfull = b_empty + 8 * kStages,
                   b_qempty = b_qfull + 16, b_sready = b_qempty + 16,
                   b_sfree = b_sready + 8 * kSBufs, b_pready = b_sfree + 8 * kSBufs,
                   b_pvdone = b_pready + 16, b_drain = b_pvdone + 16,
                   b_cready = b_drain + 16, b_kfree = b_cready + 8 * Lt::kConvSlots,
                   b_vfree = b_kfree + 8 * Lt::kConvSlots,
                   b_qsplit = b_vfree + 8 * Lt::kConvSlots, b_bkfree = b_qsplit + 16;
    constexpr int kSlots = Lt::kConvSlots;
    constexpr bool kQSplit = Lt::kQSplit;
    int *qexp = reinterpret_cast<int *>(sm + Lt::kQeOff);  // [2][kRows]
    // where the MMAs read tile j's bf16 K and V (stage s = j % kStages): the
    // TMA tile in the stage, or the ring slot j % kSlots the conversion warps
    // widened it into
    const uint32_t kconv0 = sbase + Lt::kConvOff, vconv0 = kconv0 + (KF8 ? Lt::kTileBytes : 0);
    auto k_src = [&](int st, long long j) {
        return KF8 ? kconv0 + (int)(j % kSlots) * Lt::kConvBytes : sbase + st * Lt::kStageBytes;
    };
    auto v_src = [&](int st, long long j) {
        return VF8 ? vconv0 + (int)(j % kSlots) * Lt::kConvBytes
                   : sbase + st * Lt::kStageBytes + Lt::kKBytes;
    };
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(sm + Lt::kMiscOff);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + Lt::kMiscOff + 4);
    // a ring slot is written for tile j once the MMAs of tile j - kSlots that
    // read it have completed (kfree after S, vfree after P V).  Only the
    // conversion warps wait on kfree / vfree, and they wait for every tile in
    // order: a parity wait is exact only when the barrier is at most one phase
    // behind, which a thread that skipped tiles (the producer, which runs
    // kStages tiles ahead of P V) could not ensure.
    auto slot_free = [&](uint32_t bar, long long j) {
        return j < kSlots || wait(bar + 8 * (int)(j % kSlots),
                                  (uint32_t)(((j - kSlots) / kSlots) & 1), abort_flag, p.status);
    };
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;


    // set-up that touches no global memory: it may overlap the previous
    // kernel in the stream (programmatic dependent launch)
    auto init_bars = [&]() {  // one thread
        for (int s = 0; s < kStages; ++s) {
            mbar_init(b_full + 8 * s, 1);
            mbar_init(b_empty + 8 * s, 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(b_qfull + 8 * i, 1);
            // kQSplit: the last S of the segment and every softmax warp, once
            // it has read its row's e (the next split overwrites it)
            mbar_init(b_qempty + 8 * i, kQSplit ? 1 + kSoftWarps : 1);
            mbar_init(b_pready + 8 * i, kSoftWarps);
            mbar_init(b_qsplit + 8 * i, kConvWarps);
        }
        mbar_init(b_bkfree, 1);
        for (int i = 0; i < kSBufs; ++i) {
            mbar_init(b_sready + 8 * i, 1);
            mbar_init(b_sfree + 8 * i, kSoftWarps);
        }
        mbar_init(b_pvdone, 1);
        mbar_init(b_pvdone + 8, 1);
        mbar_init(b_drain, 1);
        mbar_init(b_drain + 8, 1);
        if (Lt::kConv)
            for (int c = 0; c < kSlots; ++c) {
                mbar_init(b_cready + 8 * c, kConvWarps);
                mbar_init(b_kfree + 8 * c, 1);
                mbar_init(b_vfree + 8 * c, 1);
            }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    };
    int *len_sm = reinterpret_cast<int *>(sm + Lt::kLenOff);  // [0, 32) P, [32, 64) T
    const int lane0 = threadIdx.x & 31;
    const bool spec = p.B <= 32;
    if (threadIdx.x == 0) {
        init_bars();
        *abort_flag = 0;
    }
    if (warp == 0) {
        asm volatile(
            "tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                smem_u32(const_cast<uint32_t *>(tmem_slot))),
            "n"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    // The lengths as they read before the dependency wait (a kernel before
    // this one may still change them), one copy for the whole CTA: every
    // warp plans from the same values, and the check after the wait is the
    // same in every warp.
    if (spec && warp == kProducerWarp) {
        len_sm[lane0] = lane0 < p.B ? len_cg(p.prefix_len, lane0, p.capacity) : 0;
        len_sm[32 + lane0] = lane0 < p.B ? len_cg(p.block_len, lane0, p.max_block) : 0;
    }
    if (threadIdx.x < 64) {  // the row-sum MMA's B operand: row 0 of [8][64] bf16 ones
        const uint32_t one2 = threadIdx.x < 8 ? 0x3F803F80u : 0u;
        asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                         sbase + Lt::kOnesOff + threadIdx.x * 16),
                     "r"(one2)
                     : "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (REP) {  // both P buffers start (and, outside each copy's keys, stay) zero
        for (int i = threadIdx.x; i < 2 * Lt::kPBytes / 16; i += Lt::kThreads)
            asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                             sbase + Lt::kPOff + i * 16),
                         "r"(0u)
                         : "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == kProducerWarp && elect_one()) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_q)) : "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = *tmem_slot;

    // The plan from the lengths as they read before the dependency wait;
    // after the wait they are read again and the plan is kept only if every
    // length is unchanged.
    long long lo = 0, hi = 0, ntiles = 0;
    Walk w0 = {0, 0, 0, 1, 0, 0};
    int sP = 0, sT = 0;
    if (spec) {
        sP = len_sm[lane0];
        sT = len_sm[32 + lane0];
        ntiles = plan(p, sP, sT, lo, hi, w0) ? hi - lo : 0;
        // While the kernels before this one finish, pull the range's first
        // prefix tiles into L2 (the cache is L2-coherent: if a kernel before
        // this one writes them, the loads after the wait still see its data).
        if (warp == kProducerWarp && elect_one()) {
            Walk wp = w0;
            // the first segment's query rows (the kernel before this one may
            // be the one writing them: a prefetch only warms L2)
            if (ntiles > 0)
#pragma unroll
                for (int dp = 0; dp < Lt::kPanels; ++dp)
                    tma_prefetch_4d(&tm_q, dp * 64, wp.h * p.G, 0, wp.b);
            const int prefetch = ntiles > kLongRange ? 1 : kPrefetchTiles;
            for (long long j = 0; j < ntiles && j < prefetch && wp.t < wp.nt - 1; ++j) {
                const int tok = wp.t * kTileKeys;
#pragma unroll
                for (int dp = 0; dp < (KF8 ? 1 : Lt::kPanels); ++dp)
                    tma_prefetch_5d(&tm_k, dp * 64, wp.h, tok, wp.b, p.key_slab);
#pragma unroll
                for (int dp = 0; dp < (VF8 ? 1 : Lt::kPanels); ++dp)
                    tma_prefetch_5d(&tm_v, dp * 64, wp.h, tok, wp.b, p.value_slab);
                ++wp.t;  // stays inside the pair: its last (block) tile ends the loop
            }
        }
    }

    // Producer state and one step of its loop (tile j of the range): the
    // first steps may run before the lengths are checked (below).
    Walk wl = w0;
    int qseg = -1;
    long long nblk = 0;           // (kQSplit) block tiles whose keys were issued
    long long issued = 0, j = 0;  // tiles whose loads were issued; next tile
    bool ok = true;
    uint64_t policy = 0;
    if (warp == kProducerWarp)
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
    auto produce = [&]() {
        if (j == 0 || wl.t == 0) {  // the segment's query rows
            ++qseg;
            const int qb = qseg & 1;
            if (qseg >= 2)
                ok = ok && wait(b_qempty + 8 * qb, (uint32_t)(((qseg - 2) >> 1) & 1),
                                abort_flag, p.status);
            if (ok && elect_one()) {
                const uint32_t full = b_qfull + 8 * qb;
                const uint32_t dst = sbase + Lt::kQOff + qb * Lt::kQBytes;
                // (NC > 1) copy c at rows c 64 / NC
                mbar_arrive_expect_tx(full, NC * Lt::kPanels * p.rows_max * 128);
#pragma unroll
                for (int dp = 0; dp < Lt::kPanels; ++dp)
#pragma unroll
                    for (int c = 0; c < NC; ++c)
                        tma_4d(dst + dp * (kRows * 128) + c * (kRows / NC * 128), &tm_q, full,
                               dp * 64, wl.h * p.G, 0, wl.b);
            }
        }
        const int s = (int)(j % kStages);
        if (j >= kStages)
            ok = ok && wait(b_empty + 8 * s, (uint32_t)(((j - kStages) / kStages) & 1),
                            abort_flag, p.status);
        const bool blk = wl.t == wl.nt - 1;
        // (kQSplit) the block-key buffer is free once the S of the last block tile is done
        if (kQSplit && blk && nblk >= 1)
            ok = ok && wait(b_bkfree, (uint32_t)((nblk - 1) & 1), abort_flag, p.status);
        if (ok && elect_one()) {
            const uint32_t full = b_full + 8 * s;
            const uint32_t kdst = sbase + Lt::kStagesOff + s * Lt::kStageBytes;
            const uint32_t vdst = kdst + Lt::kKBytes;
            if (wl.t < wl.nt - 1) {
                const int tok = wl.t * kTileKeys;
                mbar_arrive_expect_tx(full, Lt::kStageBytes);
                // an e4m3 tile is one {D, 1, 64} box, a bf16 tile D / 64 swizzled panels
                if (KF8) {
                    tma_5d(kdst, &tm_k, full, 0, wl.h, tok, wl.b, p.key_slab, policy);
                } else {
#pragma unroll
                    for (int dp = 0; dp < Lt::kPanels; ++dp)
                        tma_5d(kdst + dp * 8192, &tm_k, full, dp * 64, wl.h, tok, wl.b,
                               p.key_slab, policy);
                }
                if (VF8) {
                    tma_5d(vdst, &tm_v, full, 0, wl.h, tok, wl.b, p.value_slab, policy);
                } else {
#pragma unroll
                    for (int dp = 0; dp < Lt::kPanels; ++dp)
                        tma_5d(vdst + dp * 8192, &tm_v, full, dp * 64, wl.h, tok, wl.b,
                               p.value_slab, policy);
                }
            } else if (kQSplit) {  // the block's own K (bf16) into its buffer, V into the stage
                mbar_arrive_expect_tx(full, 2 * Lt::kTileBytes);
#pragma unroll
                for (int dp = 0; dp < Lt::kPanels; ++dp) {
                    tma_4d(sbase + Lt::kBlkKOff + dp * 8192, &tm_kb, full, dp * 64, wl.h, 0,
                           wl.b);
                    tma_4d(vdst + dp * 8192, &tm_vb, full, dp * 64, wl.h, 0, wl.b);
                }
            } else {  // the block's own K / V (bf16): the operands read from the
                      // stage; ring-slot operands are loaded by the conversion warps
                mbar_arrive_expect_tx(full, (KF8 ? 0 : Lt::kTileBytes) +
                                                (VF8 ? 0 : Lt::kTileBytes));
#pragma unroll
                for (int dp = 0; dp < Lt::kPanels; ++dp) {
                    if (!KF8) tma_4d(kdst + dp * 8192, &tm_kb, full, dp * 64, wl.h, 0, wl.b);
                    if (!VF8) tma_4d(vdst + dp * 8192, &tm_vb, full, dp * 64, wl.h, 0, wl.b);
                }
            }
        }
        __syncwarp();
        if (ok && kQSplit && blk) ++nblk;
        if (ok) issued = j + 1;
        walk_next(p, wl);
        ++j;
    };

    // every input (and the workspace) may be written by the previous kernel
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // the first loads of the speculative plan go out while the lengths are
    // checked (no step here waits: fresh stages and query buffers only)
    if (spec && warp == kProducerWarp)
        while (j < ntiles && j < kStages && ok && !((j == 0 || wl.t == 0) && qseg + 1 >= 2) &&
               !(kQSplit && wl.t == wl.nt - 1 && nblk >= 1))
            produce();
    {
        const int P1 = lane0 < p.B ? len_cg(p.prefix_len, lane0, p.capacity) : 0;
        const int T1 = lane0 < p.B ? len_cg(p.block_len, lane0, p.max_block) : 0;
        if (!(spec && __all_sync(kFull, P1 == sP && T1 == sT))) {  // the same in every warp
            if (spec) {  // loads issued under the stale plan land, then the barriers restart
                if (warp == kProducerWarp) {
                    for (long long t = 0; t < issued; ++t)
                        wait(b_full + 8 * (int)t, 0u, abort_flag, p.status);
                    for (int q = 0; q <= qseg; ++q) wait(b_qfull + 8 * q, 0u, abort_flag, p.status);
                }
                __syncthreads();
                if (threadIdx.x == 0) init_bars();
                __syncthreads();
            }
            lo = hi = 0;
            w0 = {0, 0, 0, 1, 0, 0};
            ntiles = plan(p, P1, T1, lo, hi, w0) ? hi - lo : 0;
            wl = w0;
            qseg = -1;
            nblk = 0;
            issued = j = 0;
            ok = true;
        }
    }

    if (blockIdx.x == 0 && threadIdx.x == 0)
        for (int b = 0; b < p.B; ++b)
            if (p.prefix_len[b] != clamp_prefix(p, b) || p.block_len[b] != clamp_block(p, b))
                atomicOr(p.status, kStatusClamped);
    // an empty range (only when N < C) runs no loop below

    // the last loads each issuing thread started, for the abort path's drain
    long long drain_tiles = 0, drain_copy = -1;
    int drain_qseg = -1;
    if (warp == kProducerWarp) {
        // ================================ producer ===============================
        // Warp-uniform loop; one elected lane issues.  Stage s is reused once
        // the P V that read it has completed (the P V warp commits empty[s]);
        // a query buffer once the last S of the segment before last completed.
        while (j < ntiles && ok) produce();
        drain_tiles = issued;
        drain_qseg = qseg;
    } else if (warp == kMmaWarp || warp == kSWarp) {
        // ================================== MMA ==================================
        // Two issuing warps, each blocking on its own in-order stream: P V of
        // tile k once its P is in shared memory (pready), and S of tile kn once
        // its K has landed (or been widened), its segment's queries are in and
        // TMEM buffer kn % kSBufs has been read by the softmax warps (sfree).
        const uint32_t id_s = idesc(kRows, kTileKeys, 0, 0);
        const uint32_t id_pv = idesc(kRows, D, 0, 1);
        // descriptors are affine in the address: build each base once and add
        // (byte offset >> 4) for buffers and k-steps
        const uint64_t dq0 = sdesc(sbase + Lt::kQOff, 16, 1024);
        const uint64_t dk0 = sdesc(k_src(0, 0), 16, 1024);
        // (kQSplit) e4m3 operands: query parts hi / lo of buffer b at
        // kQ8Off + (2 b + part) kQ8Bytes, prefix keys in the stage, block keys (bf16)
        const uint32_t id_s8 = idesc_e4m3(kRows, kTileKeys);
        const uint64_t dq8 = sdesc(sbase + Lt::kQ8Off, 16, 1024);
        const uint64_t dk8 = sdesc(sbase + Lt::kStagesOff, 16, 1024);
        const uint64_t dkb = sdesc(sbase + Lt::kBlkKOff, 16, 1024);
        const uint64_t dv0 = sdesc(v_src(0, 0), 8192, 1024);
        const uint64_t dp0 = sdesc(sbase + Lt::kPOff, 16, 1024);
        // rounded row sums: D[64][8] += P[64][64] ones[8][64]^T, column 0 = sum of P
        const uint64_t d1 = sdesc(sbase + Lt::kOnesOff, 16, 1024);
        const uint32_t id_l = idesc(kRows, 8, 0, 0);
        bool ok = true;
        if (warp == kSWarp) {
            Walk wsn = w0;
            int qseg = -1, qcur = 0;
            for (long long kn = 0; kn < ntiles && ok; ++kn) {
                if (kn == 0 || wsn.t == 0) {
                    ++qseg;
                    qcur = qseg & 1;
                    ok = ok && wait(b_qfull + 8 * qcur, (uint32_t)((qseg >> 1) & 1), abort_flag,
                                    p.status);
                    // (kQSplit) and split into its e4m3 parts
                    if (kQSplit)
                        ok = ok && wait(b_qsplit + 8 * qcur, (uint32_t)((qseg >> 1) & 1),
                                        abort_flag, p.status);
                }
                const int s = (int)(kn % kStages);
                // the tile's K and V: landed, and widened if stored as e4m3 (kQSplit:
                // the e4m3 keys are read as they are)
                if (Lt::kConv && !kQSplit)
                    ok = ok && wait(b_cready + 8 * (int)(kn % kSlots),
                                    (uint32_t)((kn / kSlots) & 1), abort_flag, p.status);
                else
                    ok = ok && wait(b_full + 8 * s, (uint32_t)((kn / kStages) & 1), abort_flag,
                                    p.status);
                if (kn >= kSBufs)
                    ok = ok && wait(b_sfree + 8 * (int)(kn % kSBufs),
                                    (uint32_t)(((kn - kSBufs) / kSBufs) & 1), abort_flag,
                                    p.status);
                if (!ok) break;
                const bool blk_tile = wsn.t == wsn.nt - 1;
                const bool seg_end = blk_tile || (kn + 1 == ntiles);
                fence_after();
                if (elect_one()) {
                    const uint32_t dS = tmem + (uint32_t)((kn % kSBufs) * kTileKeys);
                    if (kQSplit && !blk_tile) {
                        // S = hi K^T + lo K^T: 2 x 4 MMAs of 32 e4m3 elements (32 bytes)
                        const uint64_t ah = dq8 + (uint64_t)((2 * qcur * Lt::kQ8Bytes) >> 4);
                        const uint64_t al = ah + (uint64_t)(Lt::kQ8Bytes >> 4);
                        const uint64_t b0 = dk8 + (uint64_t)((s * Lt::kStageBytes) >> 4);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_e4m3(dS, ah + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2), id_s8,
                                     kk > 0);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_e4m3(dS, al + (uint64_t)(kk * 2), b0 + (uint64_t)(kk * 2), id_s8,
                                     1u);
                    } else {
                        const uint64_t a0 = dq0 + (uint64_t)((qcur * Lt::kQBytes) >> 4);
                        const uint64_t b0 =
                            kQSplit ? dkb
                                    : dk0 + (uint64_t)((k_src(s, kn) - k_src(0, 0)) >> 4);
#pragma unroll
                        for (int kk = 0; kk < D / 16; ++kk) {
                            // panel kk / 4, then 16 elements (32 bytes) within the 128-byte row
                            const uint32_t qoff =
                                ((kk >> 2) * (kRows * 128) + (kk & 3) * 32) >> 4;
                            const uint32_t koff = ((kk >> 2) * 8192 + (kk & 3) * 32) >> 4;
                            mma(dS, a0 + qoff, b0 + koff, id_s, kk > 0);
                        }
                    }
                    mma_commit(b_sready + 8 * (int)(kn % kSBufs));
                    if (KF8 && !kQSplit) mma_commit(b_kfree + 8 * (int)(kn % kSlots));
                    if (kQSplit && blk_tile) mma_commit(b_bkfree);
                    if (seg_end) mma_commit(b_qempty + 8 * qcur);
                }
                __syncwarp();
                walk_next(p, wsn);
            }
        } else {
            Walk wm = w0;
            for (long long k = 0; k < ntiles && ok; ++k) {
                const bool first = (k == 0) || (wm.t == 0);
                ok = wait(b_pready + 8 * (int)(k & 1), (uint32_t)((k >> 1) & 1), abort_flag,
                          p.status);
                if (!ok) break;
                fence_after();
                if (elect_one()) {
                    const int s = (int)(k % kStages);
                    const uint64_t a0 = dp0 + (uint64_t)(((k & 1) * Lt::kPBytes) >> 4);
                    const uint64_t b0 = dv0 + (uint64_t)((v_src(s, k) - v_src(0, 0)) >> 4);
                    const uint32_t dO = tmem + kSBufs * kTileKeys;
#pragma unroll
                    for (int kk = 0; kk < kTileKeys / 16; ++kk)
                        mma(dO, a0 + (uint64_t)((kk * 32) >> 4),
                            b0 + (uint64_t)((kk * 2048) >> 4), id_pv,
                            (!first || kk > 0) ? 1u : 0u);
#pragma unroll
                    for (int kk = 0; kk < kTileKeys / 16; ++kk)
                        mma(dO + D, a0 + (uint64_t)((kk * 32) >> 4), d1 + (uint64_t)((kk * 32) >> 4),
                            id_l, (!first || kk > 0) ? 1u : 0u);
                    mma_commit(b_pvdone + 8 * (int)(k & 1));
                    mma_commit(b_empty + 8 * s);
                    if (VF8) mma_commit(b_vfree + 8 * (int)(k % kSlots));
                }
                __syncwarp();
                walk_next(p, wm);
            }
        }
        // all MMAs this warp issued are complete before tensor memory is freed
        // (only a timed-out run can leave any in flight)
        const uint32_t drain = b_drain + (warp == kSWarp ? 8 : 0);
        if (elect_one()) mma_commit(drain);
        __syncwarp();
        const unsigned long long t0 = globaltimer();
        while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitNs) {
        }
    } else if (kQSplit && warp >= kConvWarp0) {
        // ========================== query split (kQSplit) ========================
        // Once a segment's bf16 query rows have landed, split them into their
        // e4m3 parts for the S MMAs and record each row's e for the softmax
        // warps (qsplit).  Query buffer b is loaded again only after the S of
        // its segment and every softmax warp's read of e are done (qempty),
        // so neither the parts nor e are overwritten early.
        const int ct = threadIdx.x - kConvWarp0 * 32;
        Walk wc = w0;
        int qs = -1;
        for (long long j = 0; j < ntiles; ++j) {
            if (j == 0 || wc.t == 0) {
                ++qs;
                const int qb = qs & 1;
                if (!wait(b_qfull + 8 * qb, (uint32_t)((qs >> 1) & 1), abort_flag, p.status))
                    break;
                const uint32_t q8 = sbase + Lt::kQ8Off + 2 * qb * Lt::kQ8Bytes;
                split_q(sbase + Lt::kQOff + qb * Lt::kQBytes, q8, q8 + Lt::kQ8Bytes,
                        qexp + qb * kRows, ct);
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0) mbar_arrive(b_qsplit + 8 * qb);
            }
            walk_next(p, wc);
        }
    } else if (Lt::kConv && warp >= kConvWarp0) {
        // ============================ e4m3 -> bf16 ===============================
        // Widen every prefix tile's e4m3 K (and V) into its ring slot once it
        // has landed and the slot is free, then hand the tile to the S warp
        // (cready).  A block tile's K (V) is bf16 already: for a ring operand
        // one elected lane of the first conversion warp loads it into the slot
        // with a copy that completes on cready itself.
        const int ct = threadIdx.x - kConvWarp0 * 32;
        Walk wc = w0;
        bool ok = true;
        for (long long j = 0; j < ntiles && ok; ++j) {
            const int s = (int)(j % kStages);
            const uint32_t cready = b_cready + 8 * (int)(j % kSlots);
            ok = wait(b_full + 8 * s, (uint32_t)((j / kStages) & 1), abort_flag, p.status);
            if (!ok) break;
            if (wc.t == wc.nt - 1) {
                if (KF8) ok = slot_free(b_kfree, j);
                if (VF8) ok = ok && slot_free(b_vfree, j);
                if (!ok) break;
                if (warp == kConvWarp0) {
                    if (elect_one()) {
                        mbar_arrive_expect_tx(cready, ((KF8 ? 1 : 0) + (VF8 ? 1 : 0)) *
                                                          Lt::kTileBytes);
#pragma unroll
                        for (int dp = 0; dp < Lt::kPanels; ++dp) {
                            if (KF8)
                                tma_4d(k_src(s, j) + dp * 8192, &tm_kb, cready, dp * 64, wc.h, 0,
                                       wc.b);
                            if (VF8)
                                tma_4d(v_src(s, j) + dp * 8192, &tm_vb, cready, dp * 64, wc.h, 0,
                                       wc.b);
                        }
                    }
                    drain_copy = j;
                } else if (lane == 0) {
                    mbar_arrive(cready);
                }
                __syncwarp();
                walk_next(p, wc);
                continue;
            }
            if (KF8) {
                ok = slot_free(b_kfree, j);
                if (!ok) break;
                widen_tile<D>(sbase + s * Lt::kStageBytes, k_src(s, j), ct);
            }
            if (VF8) {
                ok = slot_free(b_vfree, j);
                if (!ok) break;
                widen_tile<D>(sbase + s * Lt::kStageBytes + Lt::kKBytes, v_src(s, j), ct);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(cready);
            walk_next(p, wc);
        }
    } else {
        // ================================ softmax ================================
        // thread (warp, lane) handles row 16 warp + lane % 16, keys of its half
        // (lane / 16) of each tile; the epilogue's O rows are read by lanes < 16
        const int row = warp * 16 + (lane & 15);
        // (REP) MMA row c 64 / NC + r holds copy c of query row r: warp w
        // holds rows of copy cp = w / (4 / NC)
        constexpr int kRowsPerCopy = kRows / NC;
        const int cp = REP ? warp / (4 / NC) : 0;
        const int qrow = REP ? row - cp * kRowsPerCopy : row;
        const int half = lane >> 4;
        // scores a thread takes per tile, and the first of them
        constexpr int kVals = 32 / NC;
        const int key0 = cp * (kTileKeys / NC) + kVals * half;
        const bool owner = lane < 16;
        const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
        Walk ws = w0;
        // l_sum: sum of the fp32 weights 2^(s - m), for the lse.  The sum of
        // the same weights as rounded to bf16 for the P V product, used for
        // the normalisation so that O / l is an exact convex combination of
        // the values (the rounding of P then moves the output by a fraction
        // of the values' spread around it, not of the values themselves), is
        // accumulated by the tensor core next to O (P times a ones column,
        // fp32), which takes its tree of adds off the softmax warps.
        float m_ref = -INFINITY, l_sum = 0.f;
        int rows_active = 0, irow = 0;
        long long seg_first = lo;
        // (kQSplit) scale of the prefix tiles' scores: S holds 2^e q.k for this row
        float row_scale = p.scale_log2;
        int qs = -1;
        for (long long k = 0; k < ntiles; ++k) {
            const bool first = (k == 0) || (ws.t == 0);
            const bool block_tile = ws.t == ws.nt - 1;
            const bool last = block_tile || (k + 1 == ntiles);
            if (first) {
                m_ref = -INFINITY;
                l_sum = 0.f;
                rows_active = p.G * ws.T;
                irow = qrow / p.G;
                seg_first = lo + k;
                if (kQSplit) {
                    ++qs;
                    const int qb = qs & 1;
                    wait(b_qsplit + 8 * qb, (uint32_t)((qs >> 1) & 1), abort_flag, p.status);
                    const int e = qexp[qb * kRows + row];
                    row_scale = p.scale_log2 * __uint_as_float((uint32_t)(127 - e) << 23);
                    __syncwarp();
                    if (lane == 0) mbar_arrive(b_qempty + 8 * qb);
                }
            }
            const int nvalid = block_tile ? ws.T : min(kTileKeys, ws.P - ws.t * kTileKeys);
            const int s = (int)(k % kStages);
            // ---- scores of tile k ----
            const bool ok_s = wait(b_sready + 8 * (int)(k % kSBufs),
                                   (uint32_t)((k / kSBufs) & 1), abort_flag, p.status);
            fence_after();
            const uint32_t s_addr = tmem + lane_base + (uint32_t)((k % kSBufs) * kTileKeys) +
                                    (uint32_t)(cp * (kTileKeys / NC));
            const bool valid_row = qrow < rows_active && ok_s;
            // keys j < lim are visible to this row; a full prefix tile needs no
            // mask (rows of other lanes are computed but never stored)
            const int lim = !valid_row ? 0 : (block_tile ? min(nvalid, irow + 1) : nvalid);
            const bool full_tile = !block_tile && nvalid == kTileKeys;
            const float scale = kQSplit && !block_tile ? row_scale : p.scale_log2;
            // The thread's 32 scores in registers (masked keys -> -inf); the
            // row's tile max decides the reference first: the segment's first
            // tile sets it, a later tile moves it (rescaling O and l) only when
            // its max is beyond the reference by more than 2^8.
            float v[kVals];
            if constexpr (kVals == 8)
                tmem_ld_half8(s_addr, v);
            else if constexpr (kVals == 16)
                tmem_ld_half16(s_addr, v);
            else
                tmem_ld_half32(s_addr, v);
            // the scores are in registers: S buffer k % kSBufs may take tile k + kSBufs
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(b_sfree + 8 * (int)(k % kSBufs));
            if (!full_tile) {
#pragma unroll
                for (int j = 0; j < kVals; j += 2) {
                    float a, b;
                    mul2(a, b, v[j], v[j + 1], scale, scale);
                    v[j] = key0 + j < lim ? a : -INFINITY;
                    v[j + 1] = key0 + j + 1 < lim ? b : -INFINITY;
                }
            }
            float mt;
            if constexpr (kVals == 8) {
                const float m = max3(max3(v[0], v[1], v[2]), max3(v[3], v[4], v[5]), fmaxf(v[6], v[7]));
                mt = full_tile ? m * scale : m;
            } else if constexpr (kVals == 16) {  // 16 -> 6 -> 2 -> 1
                const float m = fmaxf(max3(max3(v[0], v[1], v[2]), max3(v[3], v[4], v[5]),
                                           max3(v[6], v[7], v[8])),
                                      max3(max3(v[9], v[10], v[11]), max3(v[12], v[13], v[14]), v[15]));
                mt = full_tile ? m * scale : m;
            } else {  // three-input maxima: 32 -> 11 -> 4 -> 1
                float m11[11];
#pragma unroll
                for (int j = 0; j < 10; ++j) m11[j] = max3(v[3 * j], v[3 * j + 1], v[3 * j + 2]);
                m11[10] = fmaxf(v[30], v[31]);
                const float m = fmaxf(max3(max3(m11[0], m11[1], m11[2]), max3(m11[3], m11[4], m11[5]),
                                           max3(m11[6], m11[7], m11[8])),
                                      fmaxf(m11[9], m11[10]));
                mt = full_tile ? m * scale : m;
            }
            mt = fmaxf(mt, __shfl_xor_sync(kFull, mt, 16));
            if (first) {
                m_ref = mt;
            } else {
                const bool jump = valid_row && mt > m_ref + kRescaleLog2;
                if (__any_sync(kFull, jump)) {
                    // O is stable once P V of tile k-1 is done
                    wait(b_pvdone + 8 * (int)((k - 1) & 1), (uint32_t)(((k - 1) >> 1) & 1),
                         abort_flag, p.status);
                    fence_after();
                    const float alpha = jump ? ex2(m_ref - mt) : 1.f;  // m_ref -inf gives 0
                    if (jump) {
                        m_ref = mt;
                        l_sum *= alpha;
                    }
                    // O and, in the next 32 columns, the rounded row sum
#pragma unroll 1
                    for (int c = 0; c < D + 32; c += 32) {
                        float o[32];
                        const uint32_t ta = tmem + lane_base + (uint32_t)(kSBufs * kTileKeys + c);
                        tmem_ld32(ta, o);
#pragma unroll
                        for (int j = 0; j < 32; ++j) o[j] *= alpha;
                        tmem_st32(ta, o);
                    }
                }
            }
            // P = 2^(s - m) as bf16 into the swizzled P buffer (32 keys = 4
            // chunks): all exponentials first, then the packs (measured faster
            // than one loop that does both per pair); their tree sum for l
            // comes after P has been handed on
            const float mu = m_ref == -INFINITY ? 0.f : m_ref;
            if (full_tile) {
#pragma unroll
                for (int j = 0; j < kVals; j += 2)
                    fma2(v[j], v[j + 1], v[j], v[j + 1], scale, scale, -mu, -mu);
            } else {
#pragma unroll
                for (int j = 0; j < kVals; j += 2) add2(v[j], v[j + 1], v[j], v[j + 1], -mu, -mu);
            }
#pragma unroll
            for (int j = 0; j < kVals; ++j) v[j] = ex2(v[j]);
            uint32_t w[kVals / 2];
#pragma unroll
            for (int e = 0; e < kVals / 2; ++e) w[e] = pack_bf16(v[2 * e], v[2 * e + 1]);
            // P buffer (k & 1) is free once P V of tile k-2, its last reader, is done
            // (pvdone[k & 1] completes once per P V of tiles with that parity)
            if (k >= 2) wait(b_pvdone + 8 * (int)(k & 1), (uint32_t)(((k - 2) >> 1) & 1), abort_flag,
                             p.status);
            fence_after();
            const uint32_t pbuf = sbase + Lt::kPOff + (uint32_t)((k & 1) * Lt::kPBytes);
#pragma unroll
            for (int q4 = 0; q4 < kVals / 8; ++q4)
                asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                                 p_chunk_addr(pbuf, row, key0 / 8 + q4)),
                             "r"(w[4 * q4]), "r"(w[4 * q4 + 1]), "r"(w[4 * q4 + 2]),
                             "r"(w[4 * q4 + 3])
                             : "memory");
            // keys past the end of the tile may hold anything: zero their V rows
            if (nvalid < kTileKeys) {
                const uint32_t vt = v_src(s, k);
                const int nzero = (kTileKeys - nvalid) * 8 * Lt::kPanels;  // 16-byte chunks
                for (int i = threadIdx.x; i < nzero; i += kSoftWarps * 32) {
                    const int panel = i / ((kTileKeys - nvalid) * 8);
                    const int rem = i % ((kTileKeys - nvalid) * 8);
                    const int key = nvalid + rem / 8, chunk = rem % 8;
                    asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                                     vt + panel * 8192 + key * 128 + (chunk << 4)),
                                 "r"(0u)
                                 : "memory");
                }
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(b_pready + 8 * (int)(k & 1));
            if constexpr (kVals == 8) {
                l_sum += ((v[0] + v[1]) + (v[2] + v[3])) + ((v[4] + v[5]) + (v[6] + v[7]));
            } else if constexpr (kVals == 16) {
                float a0, a1, b0, b1;
                add2(a0, a1, v[0], v[1], v[8], v[9]);
                add2(b0, b1, v[2], v[3], v[10], v[11]);
                float c0, c1, d0, d1;
                add2(c0, c1, v[4], v[5], v[12], v[13]);
                add2(d0, d1, v[6], v[7], v[14], v[15]);
                add2(a0, a1, a0, a1, c0, c1);
                add2(b0, b1, b0, b1, d0, d1);
                add2(a0, a1, a0, a1, b0, b1);
                l_sum += a0 + a1;
            } else {  // the row sum is needed only for l: after P has been handed on
                // (packed adds, in the order of the tree t[j] += t[j + w])
                float t[16];
#pragma unroll
                for (int j = 0; j < 16; j += 2)
                    add2(t[j], t[j + 1], v[j], v[j + 1], v[j + 16], v[j + 17]);
#pragma unroll
                for (int wd = 8; wd > 1; wd >>= 1)
#pragma unroll
                    for (int j = 0; j < wd; j += 2)
                        add2(t[j], t[j + 1], t[j], t[j + 1], t[j + wd], t[j + wd + 1]);
                l_sum += t[0] + t[1];
            }

            // ---- end of segment: O / l and lse ----
            if (last) {
                wait(b_pvdone + 8 * (int)(k & 1), (uint32_t)((k >> 1) & 1), abort_flag, p.status);
                fence_after();
                const long long pair_first = lo + k - ws.t;
                const bool whole = (seg_first == pair_first) && block_tile;
                const int pair = ws.b * p.Hkv + ws.h;
                const size_t slot = (size_t)pair + blockIdx.x;
                const bool write = qrow < rows_active;
                // the row's sums: this thread's half plus its partner's; the
                // rounded one from the tensor core (column 0 of the row-sum
                // accumulator in the low half, column 1, zero, in the high one)
                const float l_row = l_sum + __shfl_xor_sync(kFull, l_sum, 16);
                float l_rnd;
                {
                    uint32_t r;
                    asm volatile(
                        "tcgen05.ld.sync.aligned.16x32bx2.x1.b32 {%0}, [%1], 1;\n"
                        "tcgen05.wait::ld.sync.aligned;"
                        : "=r"(r)
                        : "r"(tmem + lane_base + (uint32_t)(kSBufs * kTileKeys + D))
                        : "memory");
                    l_rnd = __uint_as_float(r);
                }
                const float l_row_rnd = l_rnd + __shfl_xor_sync(kFull, l_rnd, 16);
                const int gq = qrow % p.G;
                // this thread's columns: [64 g + 32 half, +32) for each 64-column group g
                float v[D / 2];
                tmem_ld_orow<D>(tmem + lane_base + (uint32_t)(kSBufs * kTileKeys), v);
                if constexpr (REP && Lt::kCompactXch) {
                    // The NC copies of each row through shared memory: the
                    // groups of its O row (not normalised) that the other
                    // copies combine, and its (m, l, rounded l); then thread
                    // (copy cp, row r, half) combines group cp of half `half`
                    // of query row r by log-sum-exp over the copies.
                    constexpr int kG = D / 2 / NC;  // values per group
                    constexpr int kXS = Lt::kXchStride;
                    float *xo = reinterpret_cast<float *>(sm + Lt::kXchOff);
                    float *xm = xo + 2 * kRows * kXS;
                    float *dst = xo + (half * kRows + row) * kXS;
#pragma unroll
                    for (int g = 0; g < NC; ++g) {
                        if (g == cp) continue;
                        const int slot = g < cp ? g : g - 1;
#pragma unroll
                        for (int j = 0; j < kG; j += 4)
                            *reinterpret_cast<float4 *>(dst + slot * kG + j) =
                                make_float4(v[g * kG + j], v[g * kG + j + 1], v[g * kG + j + 2],
                                            v[g * kG + j + 3]);
                    }
                    if (half == 0)
                        *reinterpret_cast<float4 *>(xm + row * 4) =
                            make_float4(m_ref, l_row, l_row_rnd, 0.f);
                    // this thread's own group, selected without a dynamic register index
                    constexpr int kDims = kG;
                    float own[kG];
#pragma unroll
                    for (int j = 0; j < kG; ++j) own[j] = v[j];
#pragma unroll
                    for (int g = 1; g < NC; ++g)
                        if (cp == g)
#pragma unroll
                            for (int j = 0; j < kG; ++j) own[j] = v[g * kG + j];
                    asm volatile("bar.sync 1, 128;" ::: "memory");
                    // group cp's dims: values [0, 32) of a half are dims 32 half + i,
                    // values [32, 64) dims 64 + 32 half + i - 32
                    const int i0 = cp * kG;
                    const int d0 = i0 < 32 ? 32 * half + i0 : 64 + 32 * half + (i0 - 32);
                    float4 ml[NC];
                    float M = -INFINITY;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        ml[c] = *reinterpret_cast<const float4 *>(xm + (c * kRowsPerCopy + qrow) * 4);
                        M = fmaxf(M, ml[c].x);
                    }
                    float L = 0.f, Lr = 0.f, o[kDims];
#pragma unroll
                    for (int j = 0; j < kDims; ++j) o[j] = 0.f;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        // a copy that saw no visible key has m = -inf and weight 0
                        const float sc = ml[c].x == -INFINITY ? 0.f : ex2(ml[c].x - M);
                        L += sc * ml[c].y;
                        Lr += sc * ml[c].z;
                        if (c == cp) {
#pragma unroll
                            for (int j = 0; j < kDims; ++j) o[j] += sc * own[j];
                        } else {
                            const float *src = xo + (half * kRows + c * kRowsPerCopy + qrow) * kXS +
                                               (cp < c ? cp : cp - 1) * kG;
#pragma unroll
                            for (int j = 0; j < kDims; j += 4) {
                                const float4 x = *reinterpret_cast<const float4 *>(src + j);
                                o[j] += sc * x.x;
                                o[j + 1] += sc * x.y;
                                o[j + 2] += sc * x.z;
                                o[j + 3] += sc * x.w;
                            }
                        }
                    }
                    const float inv = Lr > 0.f ? 1.f / Lr : 0.f;
                    const float lse = L > 0.f ? (M + __log2f(L)) * kLn2 : -INFINITY;
                    if (write) {
                        if (whole) {
                            uint16_t *orow = p.out + (((size_t)ws.b * p.max_block + irow) * p.Hq +
                                                      (size_t)ws.h * p.G + gq) * D + d0;
#pragma unroll
                            for (int j = 0; j < kDims; j += 8)
                                *reinterpret_cast<uint4 *>(orow + j) =
                                    make_uint4(pack_bf16(o[j] * inv, o[j + 1] * inv),
                                               pack_bf16(o[j + 2] * inv, o[j + 3] * inv),
                                               pack_bf16(o[j + 4] * inv, o[j + 5] * inv),
                                               pack_bf16(o[j + 6] * inv, o[j + 7] * inv));
                        } else {
                            float *prow = p.part_o + (slot * p.rows_max + qrow) * D + d0;
#pragma unroll
                            for (int j = 0; j < kDims; j += 4)
                                *reinterpret_cast<float4 *>(prow + j) =
                                    make_float4(o[j] * inv, o[j + 1] * inv, o[j + 2] * inv,
                                                o[j + 3] * inv);
                        }
                        if (cp == 0 && half == 0) {
                            if (whole)
                                p.lse[((size_t)ws.b * p.Hq + (size_t)ws.h * p.G + gq) *
                                          p.max_block +
                                      irow] = lse;
                            else
                                p.part_lse[slot * p.rows_max + qrow] = lse;
                        }
                    }
                    // the exchange area is free again once every thread has read it
                    asm volatile("bar.sync 1, 128;" ::: "memory");
                } else if constexpr (REP) {
                    // The NC copies of each row through shared memory: every
                    // copy's O row (not normalised) and its (m, l, rounded l);
                    // then thread (copy cp, row r, half) combines kDims dims of
                    // query row r, from kDims (2 cp + half), by log-sum-exp
                    // over the copies.
                    constexpr int kDims = kRowsPerCopy * D / 128;
                    float *xo = reinterpret_cast<float *>(sm + Lt::kXchOff);
                    float *xm = xo + kRows * Lt::kXchStride;
                    float *dst = xo + row * Lt::kXchStride + 32 * half;
#pragma unroll
                    for (int g = 0; g < D / 64; ++g)
#pragma unroll
                        for (int j = 0; j < 32; j += 4)
                            *reinterpret_cast<float4 *>(dst + 64 * g + j) =
                                make_float4(v[32 * g + j], v[32 * g + j + 1], v[32 * g + j + 2],
                                            v[32 * g + j + 3]);
                    if (half == 0)
                        *reinterpret_cast<float4 *>(xm + row * 4) =
                            make_float4(m_ref, l_row, l_row_rnd, 0.f);
                    asm volatile("bar.sync 1, 128;" ::: "memory");
                    const int d0 = kDims * (2 * cp + half);
                    float4 ml[NC];
                    float M = -INFINITY;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        ml[c] = *reinterpret_cast<const float4 *>(xm + (c * kRowsPerCopy + qrow) * 4);
                        M = fmaxf(M, ml[c].x);
                    }
                    float L = 0.f, Lr = 0.f, o[kDims];
#pragma unroll
                    for (int j = 0; j < kDims; ++j) o[j] = 0.f;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        // a copy that saw no visible key has m = -inf and weight 0
                        const float sc = ml[c].x == -INFINITY ? 0.f : ex2(ml[c].x - M);
                        L += sc * ml[c].y;
                        Lr += sc * ml[c].z;
                        const float *src = xo + (c * kRowsPerCopy + qrow) * Lt::kXchStride + d0;
#pragma unroll
                        for (int j = 0; j < kDims; j += 4) {
                            const float4 x = *reinterpret_cast<const float4 *>(src + j);
                            o[j] += sc * x.x;
                            o[j + 1] += sc * x.y;
                            o[j + 2] += sc * x.z;
                            o[j + 3] += sc * x.w;
                        }
                    }
                    const float inv = Lr > 0.f ? 1.f / Lr : 0.f;
                    const float lse = L > 0.f ? (M + __log2f(L)) * kLn2 : -INFINITY;
                    if (write) {
                        if (whole) {
                            uint16_t *orow = p.out + (((size_t)ws.b * p.max_block + irow) * p.Hq +
                                                      (size_t)ws.h * p.G + gq) * D + d0;
#pragma unroll
                            for (int j = 0; j < kDims; j += 8)
                                *reinterpret_cast<uint4 *>(orow + j) =
                                    make_uint4(pack_bf16(o[j] * inv, o[j + 1] * inv),
                                               pack_bf16(o[j + 2] * inv, o[j + 3] * inv),
                                               pack_bf16(o[j + 4] * inv, o[j + 5] * inv),
                                               pack_bf16(o[j + 6] * inv, o[j + 7] * inv));
                        } else {
                            float *prow = p.part_o + (slot * p.rows_max + qrow) * D + d0;
#pragma unroll
                            for (int j = 0; j < kDims; j += 4)
                                *reinterpret_cast<float4 *>(prow + j) =
                                    make_float4(o[j] * inv, o[j + 1] * inv, o[j + 2] * inv,
                                                o[j + 3] * inv);
                        }
                        if (cp == 0 && half == 0) {
                            if (whole)
                                p.lse[((size_t)ws.b * p.Hq + (size_t)ws.h * p.G + gq) *
                                          p.max_block +
                                      irow] = lse;
                            else
                                p.part_lse[slot * p.rows_max + qrow] = lse;
                        }
                    }
                    // the exchange area is free again once every thread has read it
                    asm volatile("bar.sync 1, 128;" ::: "memory");
                } else {
                const float inv = l_row_rnd > 0.f ? 1.f / l_row_rnd : 0.f;
                const float lse = l_row > 0.f ? (m_ref + __log2f(l_row)) * kLn2 : -INFINITY;
                if (write) {
                    uint16_t *orow = p.out + (((size_t)ws.b * p.max_block + irow) * p.Hq +
                                              (size_t)ws.h * p.G + gq) * D + 32 * half;
                    float *prow = p.part_o + (slot * p.rows_max + row) * D + 32 * half;
#pragma unroll
                    for (int g = 0; g < D / 64; ++g) {
                        const float *x = v + 32 * g;
                        if (whole) {
#pragma unroll
                            for (int j = 0; j < 32; j += 8)
                                *reinterpret_cast<uint4 *>(orow + 64 * g + j) =
                                    make_uint4(pack_bf16(x[j] * inv, x[j + 1] * inv),
                                               pack_bf16(x[j + 2] * inv, x[j + 3] * inv),
                                               pack_bf16(x[j + 4] * inv, x[j + 5] * inv),
                                               pack_bf16(x[j + 6] * inv, x[j + 7] * inv));
                        } else {
#pragma unroll
                            for (int j = 0; j < 32; j += 4)
                                *reinterpret_cast<float4 *>(prow + 64 * g + j) =
                                    make_float4(x[j] * inv, x[j + 1] * inv, x[j + 2] * inv,
                                                x[j + 3] * inv);
                        }
                    }
                }
                if (write && owner) {
                    if (whole)
                        p.lse[((size_t)ws.b * p.Hq + (size_t)ws.h * p.G + gq) * p.max_block +
                              irow] = lse;
                    else
                        p.part_lse[slot * p.rows_max + row] = lse;
                }
                }  // REP
                if (whole) {  // rows past the block: 0 and lse -inf
                    for (int idx = threadIdx.x; idx < (p.rows_max - rows_active) * (D / 8);
                         idx += kSoftWarps * 32) {
                        const int r = rows_active + idx / (D / 8), col = (idx % (D / 8)) * 8;
                        const int ii = r / p.G, gg = r % p.G;
                        *reinterpret_cast<uint4 *>(p.out + (((size_t)ws.b * p.max_block + ii) *
                                                                 p.Hq +
                                                             (size_t)ws.h * p.G + gg) * D + col) =
                            make_uint4(0u, 0u, 0u, 0u);
                        if (col == 0)
                            p.lse[((size_t)ws.b * p.Hq + (size_t)ws.h * p.G + gg) * p.max_block +
                                  ii] = -INFINITY;
                    }
                }
                fence_before();
            }
            walk_next(p, ws);
        }
    }
    // every MMA was waited on by the control lane and the softmax warps
    fence_before();
    __syncthreads();
    fence_after();
    if (*abort_flag) {  // a wait gave up: copies still in flight land before exit
        if (warp == kProducerWarp && elect_one()) {
            for (long long j = drain_tiles - 1; j >= 0 && j >= drain_tiles - kStages; --j)
                drain_wait(b_full + 8 * (int)(j % kStages), (uint32_t)((j / kStages) & 1));
            for (int q = drain_qseg; q >= 0 && q >= drain_qseg - 1; --q)
                drain_wait(b_qfull + 8 * (q & 1), (uint32_t)((q >> 1) & 1));
        }
        if (Lt::kConv && warp == kConvWarp0 && lane == 0 && drain_copy >= 0)
            drain_wait(b_cready + 8 * (int)(drain_copy % kSlots),
                       (uint32_t)((drain_copy / kSlots) & 1));
    }
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "n"(kTmemCols));
}

}  // namespace

// ---- split-K merge ------------------------------------------------------------
// One warp per RPW query rows of a split pair (rows w, w + 4, ... of the
// CTA's 4 RPW rows); lane l holds columns [VPL l, VPL (l+1)).  With partial s
// holding O_s / l_s and lse_s for the row:
//   out = sum_s e^(lse_s - M) O_s / l_s / sum_s e^(lse_s - M),
//   lse = M + ln sum_s e^(lse_s - M),  M = max_s lse_s,
// and rows past the block get 0 and lse -inf.  The pair's segments are found
// from the lengths before griddepcontrol.wait (the attention grid this one
// depends on started after every kernel that could write them had
// completed); the partials are read after it, SEGS segments of each of the
// RPW rows in flight at once.  SEGS x RPW trades round trips and CTAs for
// registers: at D = 128, 8 x 1 takes 116 registers a thread (4 CTAs per SM),
// 4 x 1 72 (7), 2 x 1 40 (12), 2 x 2 about the same as 4 x 1 with half the
// CTAs.
constexpr int kMergeWarps = 4;

template <int SEGS, int RPW>
constexpr int merge_min_blocks() {
    return SEGS * RPW >= 8 ? 4 : SEGS * RPW >= 4 ? 7 : 12;
}

template <int D, int SEGS, int RPW>
__global__ void __launch_bounds__(kMergeWarps * 32, merge_min_blocks<SEGS, RPW>())
    merge_kernel(const AttnParams p) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    constexpr int VPL = D / 32;
    constexpr int kRowsPerCta = kMergeWarps * RPW;
    const int rblocks = (p.rows_max + kRowsPerCta - 1) / kRowsPerCta;
    const int pair = blockIdx.x / rblocks;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row0 = (blockIdx.x % rblocks) * kRowsPerCta + warp;  // rows row0 + r * kMergeWarps
    const int b = pair / p.Hkv, h = pair % p.Hkv;
    const int C = p.num_ctas;
    // one pass: all tiles, and the tiles of the sequences before b
    long long total = 0, before = 0;
    for (int b0 = 0; b0 < p.B; b0 += 32) {
        const int nt = seq_tiles(p, b0 + lane);
        total += (long long)__reduce_add_sync(kFull, (unsigned)nt) * p.Hkv;
        before += (long long)__reduce_add_sync(kFull, b0 + lane < b ? (unsigned)nt : 0u) * p.Hkv;
    }
    const Split sp = split_from_total(p, total);
    const int nt = tiles_of(clamp_prefix(p, b));
    const long long first = before + (long long)h * nt;  // the pair's first tile
    const long long first_w = first + (long long)sp.beta * pair;
    const int c0 = cta_of_w(first_w, sp, C);
    // every CTA holds a tile when beta > 0 or N >= C, so the pair's segments
    // are those of CTAs c0 .. c1; otherwise (beta = 0) each tile is a CTA of
    // its own
    const bool contiguous = sp.beta > 0 || sp.N >= C;
    const int nseg = contiguous ? cta_of_w(first_w + nt - 1, sp, C) - c0 + 1 : nt;
    const int rows_active = p.G * clamp_block(p, b);

    // partials come from the attention grid
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (nseg <= 1) return;  // a single segment wrote its output
    uint16_t *orow[RPW];
    float *lrow[RPW];
    bool act[RPW];
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
        const int row = row0 + r * kMergeWarps;
        const int i = row / p.G, g = row % p.G;
        orow[r] = p.out + (((size_t)b * p.max_block + i) * p.Hq + (size_t)h * p.G + g) * D +
                  VPL * lane;
        lrow[r] = p.lse + ((size_t)b * p.Hq + (size_t)h * p.G + g) * p.max_block + i;
        act[r] = row < rows_active;
        if (row < p.rows_max && !act[r]) {  // rows past the block: 0 and lse -inf
            if (VPL == 4)
                *reinterpret_cast<uint2 *>(orow[r]) = make_uint2(0u, 0u);
            else
                *reinterpret_cast<uint32_t *>(orow[r]) = 0u;
            if (lane == 0) *lrow[r] = -INFINITY;
        }
    }
    float M[RPW], L[RPW], acc[RPW][VPL];
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
        M[r] = -INFINITY;
        L[r] = 0.f;
#pragma unroll
        for (int v = 0; v < VPL; ++v) acc[r][v] = 0.f;
    }
#pragma unroll 1
    for (int s0 = 0; s0 < nseg; s0 += SEGS) {
        float ls[RPW][SEGS], os[RPW][SEGS][VPL];
#pragma unroll
        for (int r = 0; r < RPW; ++r)
#pragma unroll
            for (int u = 0; u < SEGS; ++u) {
                ls[r][u] = -INFINITY;
#pragma unroll
                for (int v = 0; v < VPL; ++v) os[r][u][v] = 0.f;
                if (act[r] && s0 + u < nseg) {
                    const int c = contiguous ? c0 + s0 + u : cta_of_w(first + s0 + u, sp, C);
                    const size_t rs = ((size_t)pair + c) * p.rows_max + row0 + r * kMergeWarps;
                    ls[r][u] = __ldcg(p.part_lse + rs);
                    const float *src = p.part_o + rs * D + VPL * lane;
                    if (VPL == 4) {
                        const float4 x = __ldcg(reinterpret_cast<const float4 *>(src));
                        os[r][u][0] = x.x;
                        os[r][u][1 % VPL] = x.y;
                        os[r][u][2 % VPL] = x.z;
                        os[r][u][VPL - 1] = x.w;
                    } else {
                        const float2 x = __ldcg(reinterpret_cast<const float2 *>(src));
                        os[r][u][0] = x.x;
                        os[r][u][VPL - 1] = x.y;
                    }
                }
            }
#pragma unroll
        for (int r = 0; r < RPW; ++r) {
            float mn = M[r];
#pragma unroll
            for (int u = 0; u < SEGS; ++u) mn = fmaxf(mn, ls[r][u]);
            if (mn == -INFINITY) continue;
            const float a = __expf(M[r] - mn);  // 0 while M is -inf
            L[r] *= a;
#pragma unroll
            for (int v = 0; v < VPL; ++v) acc[r][v] *= a;
#pragma unroll
            for (int u = 0; u < SEGS; ++u) {
                const float wgt = __expf(ls[r][u] - mn);  // 0 for absent segments
                L[r] += wgt;
#pragma unroll
                for (int v = 0; v < VPL; ++v) acc[r][v] += wgt * os[r][u][v];
            }
            M[r] = mn;
        }
    }
#pragma unroll
    for (int r = 0; r < RPW; ++r) {
        if (!act[r]) continue;
        const float inv = L[r] > 0.f ? 1.f / L[r] : 0.f;
        if (VPL == 4)
            *reinterpret_cast<uint2 *>(orow[r]) =
                make_uint2(pack_bf16(acc[r][0] * inv, acc[r][1 % VPL] * inv),
                           pack_bf16(acc[r][2 % VPL] * inv, acc[r][VPL - 1] * inv));
        else
            *reinterpret_cast<uint32_t *>(orow[r]) =
                pack_bf16(acc[r][0] * inv, acc[r][VPL - 1] * inv);
        if (lane == 0) *lrow[r] = L[r] > 0.f ? M[r] + __logf(L[r]) : -INFINITY;
    }
}

// The merge variants (segments in flight x rows per warp) and their resident
// CTAs per SM, looked up once per device.
constexpr int kMergeVariants = 4;
constexpr int kMergeSegs[kMergeVariants] = {8, 4, 2, 2};
constexpr int kMergeRpw[kMergeVariants] = {1, 1, 1, 2};

template <int D>
cudaError_t merge_occupancy(int dev, int occ[kMergeVariants]) {
    static std::atomic<int> cached[64][kMergeVariants];
    if (dev < 64 && cached[dev][kMergeVariants - 1].load(std::memory_order_acquire) > 0) {
        for (int v = 0; v < kMergeVariants; ++v)
            occ[v] = cached[dev][v].load(std::memory_order_relaxed);
        return cudaSuccess;
    }
    const void *fns[kMergeVariants] = {
        reinterpret_cast<const void *>(merge_kernel<D, 8, 1>),
        reinterpret_cast<const void *>(merge_kernel<D, 4, 1>),
        reinterpret_cast<const void *>(merge_kernel<D, 2, 1>),
        reinterpret_cast<const void *>(merge_kernel<D, 2, 2>)};
    for (int v = 0; v < kMergeVariants; ++v) {
        const cudaError_t e =
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ[v], fns[v], kMergeWarps * 32, 0);
        if (e != cudaSuccess) return e;
        occ[v] = std::max(occ[v], 1);
    }
    if (dev < 64) {
        for (int v = 0; v < kMergeVariants - 1; ++v)
            cached[dev][v].store(occ[v], std::memory_order_relaxed);
        cached[dev][kMergeVariants - 1].store(occ[kMergeVariants - 1], std::memory_order_release);
    }
    return cudaSuccess;
}

template <int D, bool KF8, bool VF8, int NC = 1>
cudaError_t launch_d(const AttnParams &p, const CUtensorMap &tk, const CUtensorMap &tv,
                     const CUtensorMap &tkb, const CUtensorMap &tvb, const CUtensorMap &tq,
                     cudaStream_t stream) {
    using Lt = Layout<D, KF8, VF8, NC>;
    constexpr int smem = Lt::kBytes;
    static std::atomic<bool> configured[64];  // the smem opt-in, once per device
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(attn_kernel<D, KF8, VF8, NC>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        if (dev < 64) configured[dev].store(true, std::memory_order_release);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)p.num_ctas);
    cfg.blockDim = dim3(Lt::kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, attn_kernel<D, KF8, VF8, NC>, tk, tv, tkb, tvb, tq, p);
    if (e != cudaSuccess) return e;
    // The merge variant with the fewest estimated sequential steps: waves of
    // resident merge CTAs (at least one) times L2 round trips per row (at
    // least one), for a pair's average segment count 1 + C / (B Hkv).
    const double segs = 1.0 + (double)p.num_ctas / ((double)p.B * p.Hkv);
    int occ[kMergeVariants];
    e = merge_occupancy<D>(dev, occ);
    if (e != cudaSuccess) return e;
    int best = 0;
    double best_cost = 0.0;
    long long best_ctas = 0;
    for (int v = 0; v < kMergeVariants; ++v) {
        const int rows_per_cta = kMergeWarps * kMergeRpw[v];
        const long long ctas =
            (long long)p.B * p.Hkv * ((p.rows_max + rows_per_cta - 1) / rows_per_cta);
        const double waves = std::max(1.0, (double)ctas / ((double)occ[v] * p.num_ctas));
        const double cost = waves * std::max(1.0, segs / kMergeSegs[v]);
        if (v == 0 || cost < best_cost) {
            best = v;
            best_cost = cost;
            best_ctas = ctas;
        }
    }
    cfg.gridDim = dim3((unsigned)best_ctas);
    cfg.blockDim = dim3(kMergeWarps * 32);
    cfg.dynamicSmemBytes = 0;
    if (best == 0) return cudaLaunchKernelEx(&cfg, merge_kernel<D, 8, 1>, p);
    if (best == 1) return cudaLaunchKernelEx(&cfg, merge_kernel<D, 4, 1>, p);
    if (best == 2) return cudaLaunchKernelEx(&cfg, merge_kernel<D, 2, 1>, p);
    return cudaLaunchKernelEx(&cfg, merge_kernel<D, 2, 2>, p);
}

}  // namespace tc

int attn_grid_size(int device) {
    static std::atomic<int> sms_of[64];  // the SM count, looked up once per device
    if (device >= 0 && device < 64) {
        const int known = sms_of[device].load(std::memory_order_relaxed);
        if (known > 0) return known;
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
        return 0;
    if (device >= 0 && device < 64) sms_of[device].store(sms, std::memory_order_relaxed);
    return sms;
}

namespace {
size_t round256(size_t n) { return (n + 255) & ~size_t(255); }
}  // namespace

// header | part_o [slots][rows_max][D] | part_lse [slots][rows_max], slots =
// B * Hkv + C (the slot of a segment is pair + CTA).
size_t attn_workspace_bytes(int device, int batch, int kv_heads, int rows_max, int head_dim) {
    const int C = attn_grid_size(device);
    if (C <= 0) return 0;
    const size_t slots = (size_t)batch * kv_heads + (size_t)C;
    return kWorkspaceHeader + round256(slots * rows_max * head_dim * sizeof(float)) +
           round256(slots * rows_max * sizeof(float));
}

void attn_workspace_layout(void *workspace, int batch, int kv_heads, int rows_max, int head_dim,
                           int num_ctas, AttnParams &p) {
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    const size_t slots = (size_t)batch * kv_heads + (size_t)num_ctas;
    p.status = reinterpret_cast<int32_t *>(ws);
    size_t off = kWorkspaceHeader;
    p.part_o = reinterpret_cast<float *>(ws + off);
    off += round256(slots * rows_max * head_dim * sizeof(float));
    p.part_lse = reinterpret_cast<float *>(ws + off);
}

cudaError_t attn_launch(const AttnParams &p, int head_dim, bool keys_e4m3, bool values_e4m3,
                        const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                        const CUtensorMap &tm_kb, const CUtensorMap &tm_vb,
                        const CUtensorMap &tm_q, cudaStream_t stream) {
#define DAS_LAUNCH(D, K8, V8) tc::launch_d<D, K8, V8>(p, tm_k, tm_v, tm_kb, tm_vb, tm_q, stream)
    if (head_dim == 128) {
        if (keys_e4m3) {
            if (values_e4m3) return DAS_LAUNCH(128, true, true);
            if (p.rows_max <= 16)
                return tc::launch_d<128, true, false, 4>(p, tm_k, tm_v, tm_kb, tm_vb, tm_q, stream);
            if (p.rows_max <= 32)
                return tc::launch_d<128, true, false, 2>(p, tm_k, tm_v, tm_kb, tm_vb, tm_q, stream);
            return DAS_LAUNCH(128, true, false);
        }
        if (values_e4m3) return DAS_LAUNCH(128, false, true);
        // at most 16 (32) rows per pair: four (two) copies of the rows (see attn_kernel)
        if (p.rows_max <= 16)
            return tc::launch_d<128, false, false, 4>(p, tm_k, tm_v, tm_kb, tm_vb, tm_q, stream);
        if (p.rows_max <= 32)
            return tc::launch_d<128, false, false, 2>(p, tm_k, tm_v, tm_kb, tm_vb, tm_q, stream);
        return DAS_LAUNCH(128, false, false);
    }
    if (head_dim == 64) {
        if (keys_e4m3) return values_e4m3 ? DAS_LAUNCH(64, true, true) : DAS_LAUNCH(64, true, false);
        return values_e4m3 ? DAS_LAUNCH(64, false, true) : DAS_LAUNCH(64, false, false);
    }
#undef DAS_LAUNCH
    return cudaErrorInvalidValue;
}

}  // namespace das
