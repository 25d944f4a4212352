// das_attention.cu -- depth-asynchronous attention (Eqs. 2-3, Sec. 3.2) and the
// full-depth verify attention (Sec. 3.4) on sm_103a, tensor-core path with
// mma.sync.
//
// Work decomposition.  Each (sequence b, kv head h) pair owns nt_b =
// ceil(P_b / 64) prefix tiles and one block tile (the draft block's own keys
// under the causal mask).  All pairs' tiles are laid end to end and the
// persistent grid of C CTAs takes equal contiguous ranges of that list, so
// ragged prefix lengths balance by construction.  A CTA's range is cut into
// segments at pair boundaries.  A segment that covers a whole pair writes the
// final output.  Otherwise it writes one partial softmax state per query row
// (O / l and lse) to workspace slot p + c (p = pair index, c = CTA index:
// unique because both increase along the list).  A second kernel, launched as
// a programmatic dependent of the first, merges the pairs that were split,
//     lse = log sum_s exp(lse_s),  O = sum_s exp(lse_s - lse) O_s,
// one warp per query row with all of the row's partials loaded at once.
//
// Inside a CTA: TMA loads of 64-key K and V tiles (128-byte swizzled, two
// 64-wide panels for D = 128) run STAGES tiles ahead in a ring of shared-
// memory stages; an mbarrier per stage signals the bytes landed, and the last
// of the four warps to finish reading a stage refills it (a shared counter,
// no waiting).  Warps 0-3 compute with mma.sync m16n8k16 (bf16
// in, fp32 accumulate): S = Q K^T, fp32 online softmax in base 2, O += P V.
// Query rows of a pair are r = i * G + g (block row i, group member g); 16
// rows make an m-tile.  With one m-tile the four warps split each tile's keys
// four ways (KS = 4), with two m-tiles two ways (KS = 2), with three or four
// m-tiles every warp takes one m-tile and all 64 keys (KS = 1).  Warps that
// shared an m-tile combine their states through shared memory at the end of
// the segment.
#include <cuda_bf16.h>

#include "das_internal.h"

namespace das {
namespace {

constexpr uint32_t kFull = 0xffffffffu;
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s guard on every wait
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kThreads = kAttnThreads;  // 4 warps

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

// Wait for the phase of `parity` to complete, at most kWaitNs.  On time-out,
// or if another thread of the CTA already timed out, returns false, raises
// the CTA's abort flag and the workspace status bit; callers then skip work
// but keep the CTA's control flow (and its named barriers) intact.
__device__ __noinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity,
                                            volatile int *abort_flag, int32_t *status) {
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

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                          int32_t *status) {
#pragma unroll 1
    for (int i = 0; i < 16; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    return mbar_wait_slow(bar, parity, abort_flag, status);
}

__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int c0, int c1, int c2, int c3, int c4,
                                            uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%3, %4, %5, %6, %7}], [%2], %8;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
        "r"(c4), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int c0, int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                          uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Keep the bf16 halves of `v` whose key index is below `limit`.
__device__ __forceinline__ uint32_t keep_keys(uint32_t v, int key_lo, int limit) {
    uint32_t m = (key_lo < limit ? 0x0000ffffu : 0u) | (key_lo + 1 < limit ? 0xffff0000u : 0u);
    return v & m;
}

__device__ __forceinline__ void consumers_sync() {
    asm volatile("bar.sync 1, %0;" ::"n"(kThreads) : "memory");
}

__device__ __forceinline__ int clamp_prefix(const AttnParams &p, int b) {
    int v = p.prefix_len[b];
    return v < 0 ? 0 : (v > p.capacity ? p.capacity : v);
}
__device__ __forceinline__ int clamp_block(const AttnParams &p, int b) {
    int v = p.block_len[b];
    return v < 0 ? 0 : (v > p.max_block ? p.max_block : v);
}
__device__ __forceinline__ int tiles_of(int P) { return (P + kTileKeys - 1) / kTileKeys + 1; }

// Total tiles N, computed by one warp (all lanes get it).
__device__ long long total_tiles(const AttnParams &p) {
    int lane = threadIdx.x & 31;
    long long acc = 0;
    for (int b = lane; b < p.B; b += 32) acc += (long long)tiles_of(clamp_prefix(p, b)) * p.Hkv;
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) acc += __shfl_xor_sync(kFull, acc, d);
    return acc;
}

// Sequence b whose tiles contain list position x, and the list position of
// its first tile.  Executed by a whole warp.
__device__ void locate(const AttnParams &p, long long x, int &b_out, long long &base_out) {
    int lane = threadIdx.x & 31;
    long long run = 0;
    for (int b0 = 0; b0 < p.B; b0 += 32) {
        int b = b0 + lane;
        long long v = b < p.B ? (long long)tiles_of(clamp_prefix(p, b)) * p.Hkv : 0;
        long long inc = v;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            long long t = __shfl_up_sync(kFull, inc, d);
            if (lane >= d) inc += t;
        }
        long long total = __shfl_sync(kFull, inc, 31);
        if (run + total > x) {
            unsigned m = __ballot_sync(kFull, run + inc > x);
            int first = __ffs(m) - 1;
            long long exc = __shfl_sync(kFull, inc - v, first);
            b_out = b0 + first;
            base_out = run + exc;
            return;
        }
        run += total;
    }
    b_out = p.B;
    base_out = run;
}

// Range [c N / C, (c+1) N / C) of CTA c; the CTA whose range holds x.
__device__ __forceinline__ long long range_lo(int c, long long N, int C) {
    return (long long)c * N / C;
}
__device__ __forceinline__ int cta_of(long long x, long long N, int C) {
    return (int)(((x + 1) * (long long)C - 1) / N);
}

// Position in the tile list: sequence b, kv head h, tile t of nt.
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

template <int D>
struct Smem {
    static constexpr int kPanels = D / 64;
    static constexpr int kTileBytes = kTileKeys * D * 2;  // one of K or V
    static constexpr int kStageBytes = 2 * kTileBytes;
};

// Epilogue scratch of the KS > 1 merge: per warp 16 rows x D fp32 values,
// written into the stage of the segment's last tile (held until the epilogue
// ends; 4 x 16 x D x 4 bytes is exactly one stage).  Columns are XOR-swizzled
// by row so that the eight rows a warp writes at once fall in different banks.
__device__ __forceinline__ int epi_index(int w, int row, int col, int D) {
    return (w * 16 + row) * D + (col ^ ((row & 7) << 2));
}

template <int D, int STAGES>
constexpr int attn_smem_bytes() {
    return 1024 /* alignment slack */ + STAGES * Smem<D>::kStageBytes +
           kConsumerWarps * 16 * 2 * 4 /* m, l exchange */ + STAGES * 8 /* mbarriers */ +
           8 + 4 * STAGES /* flags, arrival counters */;
}

// Address of (key, 16-byte chunk cg) inside a 128B-swizzled [64 keys][D] tile
// stored as D/64 panels of 64 rows x 128 bytes.
__device__ __forceinline__ uint32_t swz(uint32_t tile, int key, int cg) {
    return tile + ((cg >> 3) << 13) + (key << 7) + ((((cg & 7) ^ (key & 7))) << 4);
}

// Everything one CTA keeps while walking its range.
struct Ctx {
    const AttnParams *p;
    const CUtensorMap *tm_k, *tm_v, *tm_kb, *tm_vb;
    uint8_t *stage_base;
    float *xml;
    volatile int *abort_flag;
    int *arrivals;  // [STAGES] count of warp releases of each stage
    uint32_t full0;
    long long lo, hi, N;
    int c;
    // consumer position
    Walk w;
    long long g, k;
    uint64_t policy;
};

// Load the tile at walk position wt into stage s (one thread).
template <int D>
__device__ __forceinline__ void issue_tile(const Ctx &x, const Walk &wt, int s) {
    using S = Smem<D>;
    const uint32_t full = x.full0 + 8 * s;
    const uint32_t kdst = smem_u32(x.stage_base + s * S::kStageBytes);
    const uint32_t vdst = kdst + S::kTileBytes;
    mbar_arrive_expect_tx(full, S::kStageBytes);
    if (wt.t < wt.nt - 1) {
        const int tok = wt.t * kTileKeys;
#pragma unroll
        for (int dp = 0; dp < S::kPanels; ++dp) {
            tma_load_5d(kdst + dp * 8192, x.tm_k, full, dp * 64, wt.h, tok, wt.b, x.p->key_slab,
                        x.policy);
            tma_load_5d(vdst + dp * 8192, x.tm_v, full, dp * 64, wt.h, tok, wt.b,
                        x.p->value_slab, x.policy);
        }
    } else {
#pragma unroll
        for (int dp = 0; dp < S::kPanels; ++dp) {
            tma_load_4d(kdst + dp * 8192, x.tm_kb, full, dp * 64, wt.h, 0, wt.b);
            tma_load_4d(vdst + dp * 8192, x.tm_vb, full, dp * 64, wt.h, 0, wt.b);
        }
    }
}

// Called by every warp (lane 0 acts) once it no longer reads stage s, which
// holds the tile at list position gt (walk wt).  The last of the four warps
// refills the stage with the tile STAGES positions later, without waiting.
template <int D, int STAGES>
__device__ __forceinline__ void release_stage(const Ctx &x, int s, long long gt, Walk wt) {
    if ((threadIdx.x & 31) != 0) return;
    // the counter only grows: every fourth arrival is the last of a tile
    if (atomicAdd(x.arrivals + s, 1) % kConsumerWarps != kConsumerWarps - 1) return;
    if (gt + STAGES >= x.hi || *x.abort_flag) return;
#pragma unroll
    for (int i = 0; i < STAGES; ++i) walk_next(*x.p, wt);
    // the other warps' generic-proxy reads of this stage precede their
    // arrivals; order them before the async-proxy (TMA) writes
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    issue_tile<D>(x, wt, s);
}

__device__ __forceinline__ bool seg_nonempty(int cc, long long N, int C) {
    return N >= C || range_lo(cc, N, C) != range_lo(cc + 1, N, C);
}

// Process the tiles of one segment (one pair, from x.g to the pair's block
// tile or the end of the range) with KS warps sharing each m-tile, then
// write its result.
template <int D, int STAGES, int KS>
__device__ __forceinline__ void run_segment(Ctx &x) {
    using S = Smem<D>;
    constexpr int MT = kConsumerWarps / KS;  // m-tiles
    constexpr int KPW = kTileKeys / KS;      // keys per warp in a tile
    constexpr int NT8 = KPW / 8;             // 8-key n-tiles per warp
    constexpr int KSTEPS = D / 16;
    constexpr int DTILES = D / 8;
    constexpr bool SPLIT = NT8 <= 4;  // two accumulator sets halve the S chain
    constexpr int NS2 = SPLIT ? NT8 : 1;
    const AttnParams &p = *x.p;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quad_row = lane >> 2, quad_col = (lane & 3) * 2;
    const int mw = warp % MT, kw = warp / MT;
    const int key0 = kw * KPW;

    const int sb = x.w.b, sh = x.w.h, snt = x.w.nt, sT = x.w.T;
    const int rows_active = p.G * sT;
    const long long pair_first = x.g - x.w.t;
    const long long seg_first = x.g;
    const int rowA = mw * 16 + quad_row, rowB = rowA + 8;
    const int iA = rowA / p.G, iB = rowB / p.G;

    // queries of rows rowA, rowB as m16n8k16 A fragments (0 for invalid rows)
    uint32_t qa[KSTEPS][4];
    {
        const uint16_t *qA = p.q + (((size_t)sb * p.max_block + iA) * p.Hq + (size_t)sh * p.G +
                                    rowA % p.G) * D;
        const uint16_t *qB = p.q + (((size_t)sb * p.max_block + iB) * p.Hq + (size_t)sh * p.G +
                                    rowB % p.G) * D;
        const bool vA = rowA < rows_active, vB = rowB < rows_active;
#pragma unroll
        for (int kk = 0; kk < KSTEPS; ++kk) {
            const int c0 = kk * 16 + quad_col;
            qa[kk][0] = vA ? __ldg(reinterpret_cast<const uint32_t *>(qA + c0)) : 0u;
            qa[kk][1] = vB ? __ldg(reinterpret_cast<const uint32_t *>(qB + c0)) : 0u;
            qa[kk][2] = vA ? __ldg(reinterpret_cast<const uint32_t *>(qA + c0 + 8)) : 0u;
            qa[kk][3] = vB ? __ldg(reinterpret_cast<const uint32_t *>(qB + c0 + 8)) : 0u;
        }
    }
    float o[DTILES][4];
#pragma unroll
    for (int j = 0; j < DTILES; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
    const bool compute = mw * 16 < rows_active;

    bool block_tile;
    int last_stage = 0;
    long long last_g = 0;
    Walk last_w = x.w;
    do {
        const int s = (int)(x.k % STAGES);
        const uint32_t ph = (uint32_t)((x.k / STAGES) & 1);
        const bool ok = __all_sync(kFull, mbar_wait(x.full0 + 8 * s, ph, x.abort_flag, p.status));
        block_tile = (x.w.t == snt - 1);
        const int nvalid = block_tile ? sT : min(kTileKeys, x.w.P - x.w.t * kTileKeys);
        const uint32_t kt = smem_u32(x.stage_base + s * S::kStageBytes);
        const uint32_t vt = kt + S::kTileBytes;
        if (ok && compute) {
            // ---- S = Q K^T over this warp's keys ----
            float sc[NT8][4], sc2[NS2][4];
#pragma unroll
            for (int j = 0; j < NT8; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
            for (int j = 0; j < NS2; ++j) sc2[j][0] = sc2[j][1] = sc2[j][2] = sc2[j][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk) {
#pragma unroll
                for (int jp = 0; jp < NT8 / 2; ++jp) {
                    const int key = key0 + jp * 16 + (lane & 7) + ((lane >> 4) << 3);
                    const int cg = 2 * kk + ((lane >> 3) & 1);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(swz(kt, key, cg), b0, b1, b2, b3);
                    if (SPLIT && (kk & 1)) {
                        mma_bf16(sc2[SPLIT ? 2 * jp : 0], qa[kk], b0, b1);
                        mma_bf16(sc2[SPLIT ? 2 * jp + 1 : 0], qa[kk], b2, b3);
                    } else {
                        mma_bf16(sc[2 * jp], qa[kk], b0, b1);
                        mma_bf16(sc[2 * jp + 1], qa[kk], b2, b3);
                    }
                }
            }
            // ---- scale, mask, online softmax (base 2) ----
            float tmax[2] = {-INFINITY, -INFINITY};
            const bool masked = block_tile || nvalid < key0 + KPW;
#pragma unroll
            for (int j = 0; j < NT8; ++j) {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    float v = sc[j][e];
                    if (SPLIT) v += sc2[SPLIT ? j : 0][e];
                    v *= p.scale_log2;
                    if (masked) {
                        const int key = key0 + j * 8 + quad_col + (e & 1);
                        bool valid = key < nvalid;
                        if (block_tile) valid = valid && key <= ((e >> 1) ? iB : iA);
                        v = valid ? v : -INFINITY;
                    }
                    sc[j][e] = v;
                    tmax[e >> 1] = fmaxf(tmax[e >> 1], v);
                }
            }
            float alpha[2], mu[2];
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(kFull, tmax[r], 1));
                tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(kFull, tmax[r], 2));
                const float mn = fmaxf(m_run[r], tmax[r]);
                mu[r] = mn == -INFINITY ? 0.f : mn;
                alpha[r] = ex2(m_run[r] - mu[r]);
                m_run[r] = mn;
                l_run[r] *= alpha[r];
            }
#pragma unroll
            for (int j = 0; j < DTILES; ++j) {
                o[j][0] *= alpha[0];
                o[j][1] *= alpha[0];
                o[j][2] *= alpha[1];
                o[j][3] *= alpha[1];
            }
#pragma unroll
            for (int j = 0; j < NT8; ++j) {
                sc[j][0] = ex2(sc[j][0] - mu[0]);
                sc[j][1] = ex2(sc[j][1] - mu[0]);
                sc[j][2] = ex2(sc[j][2] - mu[1]);
                sc[j][3] = ex2(sc[j][3] - mu[1]);
                l_run[0] += sc[j][0] + sc[j][1];
                l_run[1] += sc[j][2] + sc[j][3];
            }
            // ---- O += P V ----
            const bool tail = nvalid < key0 + KPW;
#pragma unroll
            for (int kk2 = 0; kk2 < KPW / 16; ++kk2) {
                const int kb = key0 + kk2 * 16;
                const uint32_t pa[4] = {pack_bf16(sc[2 * kk2][0], sc[2 * kk2][1]),
                                        pack_bf16(sc[2 * kk2][2], sc[2 * kk2][3]),
                                        pack_bf16(sc[2 * kk2 + 1][0], sc[2 * kk2 + 1][1]),
                                        pack_bf16(sc[2 * kk2 + 1][2], sc[2 * kk2 + 1][3])};
#pragma unroll
                for (int dp = 0; dp < DTILES / 2; ++dp) {
                    const int key = kb + (lane & 7) + (((lane >> 3) & 1) << 3);
                    const int cg = 2 * dp + (lane >> 4);
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_t(swz(vt, key, cg), b0, b1, b2, b3);
                    if (tail) {  // keys past the end may hold anything: zero them
                        const int k0 = kb + quad_col;
                        b0 = keep_keys(b0, k0, nvalid);
                        b1 = keep_keys(b1, k0 + 8, nvalid);
                        b2 = keep_keys(b2, k0, nvalid);
                        b3 = keep_keys(b3, k0 + 8, nvalid);
                    }
                    mma_bf16(o[2 * dp], pa, b0, b1);
                    mma_bf16(o[2 * dp + 1], pa, b2, b3);
                }
            }
        }
        __syncwarp();
        last_stage = s;
        last_g = x.g;
        last_w = x.w;
        // with KS > 1 the segment's last stage becomes the epilogue scratch:
        // it is released after the epilogue
        if (KS == 1 || !(block_tile || x.g + 1 == x.hi)) release_stage<D, STAGES>(x, s, x.g, x.w);
        ++x.k;
        ++x.g;
        walk_next(p, x.w);
    } while (!block_tile && x.g < x.hi);

    // ------------------------------ segment result ------------------------------
    const bool whole = (seg_first == pair_first) && block_tile;
    const int pair = sb * p.Hkv + sh;
    const size_t slot = (size_t)pair + x.c;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        l_run[r] += __shfl_xor_sync(kFull, l_run[r], 1);
        l_run[r] += __shfl_xor_sync(kFull, l_run[r], 2);
    }
    if (KS == 1) {
        // each warp owns its m-tile: write from registers
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int row = r == 0 ? rowA : rowB;
            if (row >= rows_active) continue;
            const float f = l_run[r] > 0.f ? 1.f / l_run[r] : 0.f;
            const float lse = l_run[r] > 0.f ? (m_run[r] + __log2f(l_run[r])) * kLn2 : -INFINITY;
            const int i = row / p.G, g = row % p.G;
            if (whole) {
                uint16_t *orow = p.out + (((size_t)sb * p.max_block + i) * p.Hq +
                                          (size_t)sh * p.G + g) * D;
#pragma unroll
                for (int j = 0; j < DTILES; ++j)
                    *reinterpret_cast<uint32_t *>(orow + j * 8 + quad_col) =
                        pack_bf16(o[j][2 * r] * f, o[j][2 * r + 1] * f);
                if ((lane & 3) == 0)
                    p.lse[((size_t)sb * p.Hq + (size_t)sh * p.G + g) * p.max_block + i] = lse;
            } else {
                float *prow = p.part_o + (slot * p.rows_max + row) * D;
#pragma unroll
                for (int j = 0; j < DTILES; ++j)
                    *reinterpret_cast<float2 *>(prow + j * 8 + quad_col) =
                        make_float2(o[j][2 * r] * f, o[j][2 * r + 1] * f);
                if ((lane & 3) == 0) p.part_lse[slot * p.rows_max + row] = lse;
            }
        }
    } else {
        // exchange (m, l) between the KS warps of an m-tile, scale each warp's
        // O by exp2(m - M) / L into its own region, then sum the regions.
        // A warp may run ahead by up to STAGES tiles: wait until every warp
        // has left the previous segment's use of xml and epi.
        consumers_sync();
        if ((lane & 3) == 0) {
            x.xml[(warp * 16 + quad_row) * 2 + 0] = m_run[0];
            x.xml[(warp * 16 + quad_row) * 2 + 1] = l_run[0];
            x.xml[(warp * 16 + quad_row + 8) * 2 + 0] = m_run[1];
            x.xml[(warp * 16 + quad_row + 8) * 2 + 1] = l_run[1];
        }
        consumers_sync();
        float *epi = reinterpret_cast<float *>(x.stage_base + last_stage * S::kStageBytes);
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int rr = quad_row + 8 * r;
            float M = -INFINITY;
#pragma unroll
            for (int k2 = 0; k2 < KS; ++k2) M = fmaxf(M, x.xml[((mw + k2 * MT) * 16 + rr) * 2]);
            const float Mu = M == -INFINITY ? 0.f : M;
            float L = 0.f;
#pragma unroll
            for (int k2 = 0; k2 < KS; ++k2) {
                const int ww = mw + k2 * MT;
                L += ex2(x.xml[(ww * 16 + rr) * 2] - Mu) * x.xml[(ww * 16 + rr) * 2 + 1];
            }
            const float f = L > 0.f ? ex2(m_run[r] - Mu) / L : 0.f;
#pragma unroll
            for (int j = 0; j < DTILES; ++j)
                *reinterpret_cast<float2 *>(epi + epi_index(warp, rr, j * 8 + quad_col, D)) =
                    make_float2(o[j][2 * r] * f, o[j][2 * r + 1] * f);
        }
        consumers_sync();
        constexpr int C4 = D / 4;
        for (int idx = threadIdx.x; idx < MT * 16 * C4; idx += kThreads) {
            const int row = idx / C4, c4 = idx % C4;
            if (row >= rows_active) continue;
            const int mt = row >> 4, rr = row & 15;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            float M = -INFINITY;
#pragma unroll
            for (int k2 = 0; k2 < KS; ++k2) {
                const int ww = mt + k2 * MT;
                const float4 v =
                    *reinterpret_cast<const float4 *>(epi + epi_index(ww, rr, 4 * c4, D));
                acc.x += v.x;
                acc.y += v.y;
                acc.z += v.z;
                acc.w += v.w;
                M = fmaxf(M, x.xml[(ww * 16 + rr) * 2]);
            }
            const int i = row / p.G, g = row % p.G;
            float lse = -INFINITY;
            if (c4 == 0) {
                const float Mu = M == -INFINITY ? 0.f : M;
                float L = 0.f;
#pragma unroll
                for (int k2 = 0; k2 < KS; ++k2) {
                    const int ww = mt + k2 * MT;
                    L += ex2(x.xml[(ww * 16 + rr) * 2] - Mu) * x.xml[(ww * 16 + rr) * 2 + 1];
                }
                lse = L > 0.f ? (Mu + __log2f(L)) * kLn2 : -INFINITY;
            }
            if (whole) {
                uint16_t *orow = p.out + (((size_t)sb * p.max_block + i) * p.Hq +
                                          (size_t)sh * p.G + g) * D;
                *reinterpret_cast<uint2 *>(orow + 4 * c4) =
                    make_uint2(pack_bf16(acc.x, acc.y), pack_bf16(acc.z, acc.w));
                if (c4 == 0)
                    p.lse[((size_t)sb * p.Hq + (size_t)sh * p.G + g) * p.max_block + i] = lse;
            } else {
                *reinterpret_cast<float4 *>(p.part_o + (slot * p.rows_max + row) * D + 4 * c4) =
                    acc;
                if (c4 == 0) p.part_lse[slot * p.rows_max + row] = lse;
            }
        }
        release_stage<D, STAGES>(x, last_stage, last_g, last_w);
    }

    if (whole) {
        // rows past the block are 0 with lse -inf
        for (int idx = threadIdx.x; idx < (p.rows_max - rows_active) * (D / 2); idx += kThreads) {
            const int row = rows_active + idx / (D / 2), col = (idx % (D / 2)) * 2;
            const int i = row / p.G, g = row % p.G;
            *reinterpret_cast<uint32_t *>(p.out + (((size_t)sb * p.max_block + i) * p.Hq +
                                                   (size_t)sh * p.G + g) * D + col) = 0u;
            if (col == 0)
                p.lse[((size_t)sb * p.Hq + (size_t)sh * p.G + g) * p.max_block + i] = -INFINITY;
        }
        return;
    }
}

template <int D, int STAGES>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    attn_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                const __grid_constant__ CUtensorMap tm_kb,
                const __grid_constant__ CUtensorMap tm_vb, const AttnParams p) {
    using S = Smem<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    Ctx x;
    x.p = &p;
    x.tm_k = &tm_k;
    x.tm_v = &tm_v;
    x.tm_kb = &tm_kb;
    x.tm_vb = &tm_vb;
    x.stage_base = smem;
    x.xml = reinterpret_cast<float *>(smem + STAGES * S::kStageBytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(x.xml + kConsumerWarps * 16 * 2);
    x.abort_flag = reinterpret_cast<volatile int *>(bars + STAGES);
    x.arrivals = const_cast<int *>(x.abort_flag) + 2;
    x.full0 = smem_u32(bars);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(x.full0 + 8 * s, 1);
            x.arrivals[s] = 0;
        }
        *x.abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x == 32) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
    }
    __syncthreads();

    // This CTA's range [lo, hi) of the tile list and its first position.
    x.c = blockIdx.x;
    const int lane = threadIdx.x & 31;
    long long base;
    if (p.B <= 32) {
        // one load of the lengths per warp; everything else by shuffles
        const int rawP = lane < p.B ? __ldg(p.prefix_len + lane) : 0;
        const int rawT = lane < p.B ? __ldg(p.block_len + lane) : 0;
        const int Pl = rawP < 0 ? 0 : (rawP > p.capacity ? p.capacity : rawP);
        const int Tl = rawT < 0 ? 0 : (rawT > p.max_block ? p.max_block : rawT);
        if (x.c == 0 && threadIdx.x < 32 && __any_sync(kFull, rawP != Pl || rawT != Tl) &&
            lane == 0)
            atomicOr(p.status, kStatusClamped);
        const long long v = lane < p.B ? (long long)tiles_of(Pl) * p.Hkv : 0;
        long long inc = v;
#pragma unroll
        for (int d = 1; d < 32; d <<= 1) {
            const long long t = __shfl_up_sync(kFull, inc, d);
            if (lane >= d) inc += t;
        }
        x.N = __shfl_sync(kFull, inc, 31);
        x.lo = range_lo(x.c, x.N, p.num_ctas);
        x.hi = range_lo(x.c + 1, x.N, p.num_ctas);
        if (x.lo >= x.hi) return;
        const int first = __ffs(__ballot_sync(kFull, inc > x.lo)) - 1;
        base = __shfl_sync(kFull, inc - v, first);
        x.w.b = first;
        x.w.P = __shfl_sync(kFull, Pl, first);
        x.w.T = __shfl_sync(kFull, Tl, first);
        x.w.nt = tiles_of(x.w.P);
    } else {
        x.N = total_tiles(p);
        x.lo = range_lo(x.c, x.N, p.num_ctas);
        x.hi = range_lo(x.c + 1, x.N, p.num_ctas);
        if (x.c == 0 && threadIdx.x == 0) {
            for (int b = 0; b < p.B; ++b)
                if (p.prefix_len[b] != clamp_prefix(p, b) || p.block_len[b] != clamp_block(p, b))
                    atomicOr(p.status, kStatusClamped);
        }
        if (x.lo >= x.hi) return;
        locate(p, x.lo, x.w.b, base);
        x.w.P = x.w.T = x.w.nt = 0;
        walk_load_seq(p, x.w);
    }
    {
        const long long off = x.lo - base;
        x.w.h = (int)(off / x.w.nt);
        x.w.t = (int)(off % x.w.nt);
    }
    x.g = x.lo;
    x.k = 0;
    // the merge grid may start loading as SMs free up; it waits for this grid
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(x.policy));
    if (threadIdx.x == 0) {
        Walk wt = x.w;
        for (int i = 0; i < STAGES && x.lo + i < x.hi; ++i) {
            issue_tile<D>(x, wt, i);
            walk_next(p, wt);
        }
    }
    while (x.g < x.hi) {
        const int rows = p.G * x.w.T;
        if (rows <= 16)
            run_segment<D, STAGES, 4>(x);
        else if (rows <= 32)
            run_segment<D, STAGES, 2>(x);
        else
            run_segment<D, STAGES, 1>(x);
    }
}

// Merge the partials of every pair that more than one CTA worked on.  Grid:
// pairs x ceil(rows_max / 4) CTAs of 4 warps, one warp per query row.
template <int D>
__global__ void __launch_bounds__(kThreads) merge_kernel(const AttnParams p) {
    // partials come from the attention grid this grid depends on
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int rblocks = (p.rows_max + kConsumerWarps - 1) / kConsumerWarps;
    const int pair = blockIdx.x / rblocks;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = (blockIdx.x % rblocks) * kConsumerWarps + warp;
    const int b = pair / p.Hkv, h = pair % p.Hkv;
    const int C = p.num_ctas;
    // total tiles N and the list position of this pair's first tile
    long long N = 0, before = 0;
    for (int b0 = 0; b0 < p.B; b0 += 32) {
        const int bb = b0 + lane;
        const long long v = bb < p.B ? (long long)tiles_of(clamp_prefix(p, bb)) * p.Hkv : 0;
        N += v;
        if (bb < b) before += v;
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        N += __shfl_xor_sync(kFull, N, d);
        before += __shfl_xor_sync(kFull, before, d);
    }
    const int nt = tiles_of(clamp_prefix(p, b));
    const long long first = before + (long long)h * nt;
    const int c0 = cta_of(first, N, C), c1 = cta_of(first + nt - 1, N, C);
    int nseg = c1 - c0 + 1;
    if (N < C) {
        nseg = 0;
        for (int cc = c0; cc <= c1; ++cc) nseg += seg_nonempty(cc, N, C);
    }
    if (nseg <= 1 || row >= p.rows_max) return;  // single segment: written directly
    const int i = row / p.G, g = row % p.G;
    uint16_t *orow = p.out + (((size_t)b * p.max_block + i) * p.Hq + (size_t)h * p.G + g) * D;
    float *lrow = p.lse + ((size_t)b * p.Hq + (size_t)h * p.G + g) * p.max_block + i;
    constexpr int VPL = D / 32;
    if (row >= p.G * clamp_block(p, b)) {
        if (VPL == 4)
            *reinterpret_cast<uint2 *>(orow + 4 * lane) = make_uint2(0u, 0u);
        else
            *reinterpret_cast<uint32_t *>(orow + 2 * lane) = 0u;
        if (lane == 0) *lrow = -INFINITY;
        return;
    }
    const float *plse = p.part_lse + row;
    const float *po = p.part_o + (size_t)row * D + VPL * lane;
    const size_t sstride = (size_t)p.rows_max;  // per slot, in rows
    float M = -INFINITY;
    for (int cc = c0 + lane; cc <= c1; cc += 32)
        if (seg_nonempty(cc, N, C)) M = fmaxf(M, plse[((size_t)pair + cc) * sstride]);
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, d));
    float L = 0.f;
    float acc[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) acc[v] = 0.f;
    for (int base = c0; base <= c1; base += 32) {
        const int cc = base + lane;
        float wl = 0.f;
        if (cc <= c1 && seg_nonempty(cc, N, C)) wl = __expf(plse[((size_t)pair + cc) * sstride] - M);
        L += wl;
        const int n = min(32, c1 - base + 1);
        int t = 0;
        for (; t + 8 <= n; t += 8) {
            float w8[8];
            float vals[8][VPL];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                w8[u] = __shfl_sync(kFull, wl, t + u);
                const float *src = po + ((size_t)pair + base + t + u) * sstride * D;
                if (VPL == 4) {
                    const float4 x4 = *reinterpret_cast<const float4 *>(src);
                    vals[u][0] = x4.x;
                    vals[u][1 % VPL] = x4.y;
                    vals[u][2 % VPL] = x4.z;
                    vals[u][VPL - 1] = x4.w;
                } else {
                    const float2 x2 = *reinterpret_cast<const float2 *>(src);
                    vals[u][0] = x2.x;
                    vals[u][VPL - 1] = x2.y;
                }
            }
#pragma unroll
            for (int u = 0; u < 8; ++u)
                if (w8[u] != 0.f)  // empty CTAs (only when N < C) carry weight 0
#pragma unroll
                    for (int v = 0; v < VPL; ++v) acc[v] += w8[u] * vals[u][v];
        }
        for (; t < n; ++t) {
            const float wgt = __shfl_sync(kFull, wl, t);
            if (wgt == 0.f) continue;
            const float *src = po + ((size_t)pair + base + t) * sstride * D;
#pragma unroll
            for (int v = 0; v < VPL; ++v) acc[v] += wgt * src[v];
        }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) L += __shfl_xor_sync(kFull, L, d);
    const float inv = 1.f / L;
    if (VPL == 4)
        *reinterpret_cast<uint2 *>(orow + 4 * lane) =
            make_uint2(pack_bf16(acc[0] * inv, acc[1 % VPL] * inv),
                       pack_bf16(acc[2 % VPL] * inv, acc[VPL - 1] * inv));
    else
        *reinterpret_cast<uint32_t *>(orow + 2 * lane) = pack_bf16(acc[0] * inv, acc[VPL - 1] * inv);
    if (lane == 0) *lrow = M + __logf(L);
}

template <int D>
constexpr int kStages = (D == 128) ? 3 : 6;

template <int D>
cudaError_t merge_launch_d(const AttnParams &p, cudaStream_t stream);

template <int D>
cudaError_t launch_d(const AttnParams &p, const CUtensorMap &tk, const CUtensorMap &tv,
                     const CUtensorMap &tkb, const CUtensorMap &tvb, cudaStream_t stream) {
    constexpr int ST = kStages<D>;
    constexpr int smem = attn_smem_bytes<D, ST>();
    static bool configured[64] = {false};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 64 && !configured[dev]) {
        e = cudaFuncSetAttribute(attn_kernel<D, ST>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 smem);
        if (e != cudaSuccess) return e;
        configured[dev] = true;
    }
    attn_kernel<D, ST><<<p.num_ctas, kThreads, smem, stream>>>(tk, tv, tkb, tvb, p);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return merge_launch_d<D>(p, stream);
}

template <int D>
cudaError_t merge_launch_d(const AttnParams &p, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(p.B * p.Hkv * ((p.rows_max + kConsumerWarps - 1) / kConsumerWarps)));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, merge_kernel<D>, p);
}

}  // namespace

int attn_grid_size(int device) {
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
        return 0;
    return sms * kCtasPerSm;
}

size_t attn_workspace_bytes(int device, int batch, int kv_heads, int rows_max, int head_dim) {
    const int C = attn_grid_size(device);
    if (C <= 0) return 0;
    const size_t slots = (size_t)batch * kv_heads + (size_t)C;
    size_t bytes = kWorkspaceHeader;
    bytes += slots * rows_max * head_dim * sizeof(float);
    bytes = (bytes + 255) & ~size_t(255);
    bytes += slots * rows_max * sizeof(float);
    return (bytes + 255) & ~size_t(255);
}

void attn_workspace_layout(void *workspace, int batch, int kv_heads, int rows_max, int head_dim,
                           int num_ctas, AttnParams &p) {
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    const size_t slots = (size_t)batch * kv_heads + (size_t)num_ctas;
    p.status = reinterpret_cast<int32_t *>(ws);
    size_t off = kWorkspaceHeader;
    p.part_o = reinterpret_cast<float *>(ws + off);
    off += slots * rows_max * head_dim * sizeof(float);
    off = (off + 255) & ~size_t(255);
    p.part_lse = reinterpret_cast<float *>(ws + off);
}

cudaError_t attn_merge_launch(const AttnParams &p, int head_dim, cudaStream_t stream) {
    if (head_dim == 128) return merge_launch_d<128>(p, stream);
    if (head_dim == 64) return merge_launch_d<64>(p, stream);
    return cudaErrorInvalidValue;
}

cudaError_t attn_launch(const AttnParams &p, int head_dim, const CUtensorMap &tm_k,
                        const CUtensorMap &tm_v, const CUtensorMap &tm_kb,
                        const CUtensorMap &tm_vb, cudaStream_t stream) {
    if (head_dim == 128) return launch_d<128>(p, tm_k, tm_v, tm_kb, tm_vb, stream);
    if (head_dim == 64) return launch_d<64>(p, tm_k, tm_v, tm_kb, tm_vb, stream);
    return cudaErrorInvalidValue;
}

}  // namespace das
