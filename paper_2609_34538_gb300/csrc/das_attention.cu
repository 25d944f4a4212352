// das_attention.cu -- depth-asynchronous attention (Eqs. 2-3, Sec. 3.2) and the
// full-depth verify attention (Sec. 3.4) on sm_103a.
//
// Work decomposition.  Each (sequence b, kv head h) pair owns nt_b =
// ceil(P_b / 64) prefix tiles and one block tile (the draft block's own keys
// under the causal mask).  All pairs' tiles are laid end to end and the
// persistent grid of C CTAs takes equal contiguous ranges of that list, so
// ragged prefix lengths balance by construction.  A CTA's range is cut into
// segments at pair boundaries; each segment yields one partial softmax state
// (O / l, lse) per query row, written to workspace slot p + c (p = pair
// index, c = CTA index: unique because both increase along the list).  A
// segment that covers a whole pair writes the final output directly.  A
// second kernel merges the partials of the pairs that were split:
//     lse = log sum_s exp(lse_s),  O = sum_s exp(lse_s - lse) O_s.
//
// Inside a CTA: thread 0 issues TMA loads of 64-key K and V tiles (128-byte
// swizzled, two 64-wide panels for D = 128) STAGES tiles ahead into a ring of
// shared-memory stages guarded by mbarriers (full: bytes landed; empty: all
// four warps done reading).  Warps 0-3 compute with mma.sync m16n8k16
// (bf16 in, fp32 accumulate): S = Q K^T, fp32 online softmax in base 2,
// O += P V.  Query rows of a pair are r = i * G + g (block row i, group
// member g); 16 rows make an m-tile.  With one m-tile the four warps split
// each tile's keys four ways, with two m-tiles two ways, with three or four
// m-tiles every warp takes one m-tile and all 64 keys.  Warps that shared an
// m-tile combine their states through shared memory at the segment's end.
#include <cuda_bf16.h>

#include "das_internal.h"

namespace das {
namespace {

constexpr uint32_t kFull = 0xffffffffu;
constexpr unsigned long long kWaitNs = 2000000000ull;  // 2 s guard on every wait
constexpr float kLn2 = 0.6931471805599453f;

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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                          int32_t *status) {
    if (*abort_flag) return false;
    if (mbar_try_wait(bar, parity)) return true;
    unsigned long long t0 = globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((it & 255u) == 0) {
            if (*abort_flag) return false;
            if (globaltimer() - t0 > kWaitNs) {
                *abort_flag = 1;
                atomicOr(status, kStatusWaitTimeout);
                return false;
            }
        }
    }
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

__device__ __forceinline__ void named_bar_sync(int id, int threads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
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

// CTA whose range holds list position x (ranges are [c N / C, (c+1) N / C)).
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
    static constexpr int kEpiBytes = 2 * 16 * D * 4;  // two m-tiles of fp32 rows
};

template <int D, int STAGES>
constexpr int attn_smem_bytes() {
    return 1024 /* alignment slack */ + STAGES * Smem<D>::kStageBytes + Smem<D>::kEpiBytes +
           kConsumerWarps * 16 * 2 * 4 /* m, l exchange */ + 2 * STAGES * 8 /* mbarriers */ +
           16 /* abort flag */;
}

// Address of (key, 16-byte chunk cg) inside a 128B-swizzled [64 keys][D] tile
// stored as D/64 panels of 64 rows x 128 bytes.
__device__ __forceinline__ uint32_t swz(uint32_t tile, int key, int cg) {
    return tile + ((cg >> 3) << 13) + (key << 7) + ((((cg & 7) ^ (key & 7))) << 4);
}

template <int D, int STAGES>
__global__ void __launch_bounds__(kAttnThreads, kCtasPerSm)
    attn_kernel(const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
                const __grid_constant__ CUtensorMap tm_kb, const __grid_constant__ CUtensorMap tm_vb,
                const AttnParams p) {
    constexpr int KSTEPS = D / 16;    // k-steps over head_dim in S = Q K^T
    constexpr int DTILES = D / 8;     // n-tiles over head_dim in O
    using S = Smem<D>;

    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~uintptr_t(1023));
    uint8_t *stage_base = smem;
    float *epi = reinterpret_cast<float *>(smem + STAGES * S::kStageBytes);
    float *xml = reinterpret_cast<float *>(smem + STAGES * S::kStageBytes + S::kEpiBytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(xml + kConsumerWarps * 16 * 2);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bars + 2 * STAGES);
    const uint32_t full0 = smem_u32(bars), empty0 = smem_u32(bars + STAGES);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, kConsumerWarps);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (threadIdx.x == 32) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_k)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tm_v)) : "memory");
    }
    __syncthreads();

    // This CTA's range [lo, hi) of the tile list.
    const long long N = total_tiles(p);
    const int C = p.num_ctas, c = blockIdx.x;
    const long long lo = (long long)c * N / C, hi = (long long)(c + 1) * N / C;
    if (c == 0 && threadIdx.x == 0) {
        for (int b = 0; b < p.B; ++b)
            if (p.prefix_len[b] != clamp_prefix(p, b) || p.block_len[b] != clamp_block(p, b))
                atomicOr(p.status, kStatusClamped);
    }
    if (lo >= hi) return;
    Walk w;
    {
        long long base;
        locate(p, lo, w.b, base);
        w.P = w.T = w.nt = 0;
        walk_load_seq(p, w);
        long long off = lo - base;
        w.h = (int)(off / w.nt);
        w.t = (int)(off % w.nt);
    }

    // ---------------- loads: thread 0 runs STAGES tiles ahead ----------------
    Walk pw = w;         // position of the next tile to load
    long long pg = lo;   // its list position
    uint64_t policy = 0;
    if (threadIdx.x == 0)
        asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
    auto issue_next = [&]() {
        const long long j = pg - lo;
        const int s = (int)(j % STAGES);
        const uint32_t ph = (uint32_t)((j / STAGES) & 1);
        if (!mbar_wait(empty0 + 8 * s, ph ^ 1u, abort_flag, p.status)) {
            pg = hi;
            return;
        }
        const uint32_t full = full0 + 8 * s;
        const uint32_t kdst = smem_u32(stage_base + s * S::kStageBytes);
        const uint32_t vdst = kdst + S::kTileBytes;
        mbar_arrive_expect_tx(full, S::kStageBytes);
        if (pw.t < pw.nt - 1) {
            const int tok = pw.t * kTileKeys;
#pragma unroll
            for (int dp = 0; dp < S::kPanels; ++dp) {
                tma_load_5d(kdst + dp * 8192, &tm_k, full, dp * 64, pw.h, tok, pw.b, p.key_slab,
                            policy);
                tma_load_5d(vdst + dp * 8192, &tm_v, full, dp * 64, pw.h, tok, pw.b, p.value_slab,
                            policy);
            }
        } else {
#pragma unroll
            for (int dp = 0; dp < S::kPanels; ++dp) {
                tma_load_4d(kdst + dp * 8192, &tm_kb, full, dp * 64, pw.h, 0, pw.b);
                tma_load_4d(vdst + dp * 8192, &tm_vb, full, dp * 64, pw.h, 0, pw.b);
            }
        }
        walk_next(p, pw);
        ++pg;
    };
    if (threadIdx.x == 0)
        for (int i = 0; i < STAGES && pg < hi; ++i) issue_next();

    // ---------------- consumers: warps 0..3 ----------------
    const int quad_row = lane >> 2, quad_col = (lane & 3) * 2;
    uint32_t qa[KSTEPS][4];
    float o[DTILES][4];
    float m_run[2], l_run[2];
    int mt_pad = 1, ks = 4, mw = 0, kw = 0, kpw = 16;
    int rowA = 0, rowB = 0, iA = 0, iB = 0, rows_active = 0;
    long long seg_first = lo;  // list position where the current segment began
    long long pair_first = 0;  // list position of the current pair's first tile

    auto begin_segment = [&](long long g) {
        rows_active = p.G * w.T;
        mt_pad = rows_active <= 16 ? 1 : (rows_active <= 32 ? 2 : 4);
        ks = kConsumerWarps / mt_pad;
        mw = warp % mt_pad;
        kw = warp / mt_pad;
        kpw = kTileKeys / ks;
        rowA = mw * 16 + quad_row;
        rowB = rowA + 8;
        iA = rowA / p.G;
        iB = rowB / p.G;
        seg_first = g;
        pair_first = g - w.t;
        // queries of rows rowA, rowB as m16n8k16 A fragments (0 for invalid rows)
        const uint16_t *qA = p.q + (((size_t)w.b * p.max_block + iA) * p.Hq + (size_t)w.h * p.G +
                                    rowA % p.G) * D;
        const uint16_t *qB = p.q + (((size_t)w.b * p.max_block + iB) * p.Hq + (size_t)w.h * p.G +
                                    rowB % p.G) * D;
        const bool vA = rowA < rows_active, vB = rowB < rows_active;
#pragma unroll
        for (int kk = 0; kk < KSTEPS; ++kk) {
            const int c0 = kk * 16 + quad_col;
            qa[kk][0] = vA ? *reinterpret_cast<const uint32_t *>(qA + c0) : 0u;
            qa[kk][1] = vB ? *reinterpret_cast<const uint32_t *>(qB + c0) : 0u;
            qa[kk][2] = vA ? *reinterpret_cast<const uint32_t *>(qA + c0 + 8) : 0u;
            qa[kk][3] = vB ? *reinterpret_cast<const uint32_t *>(qB + c0 + 8) : 0u;
        }
#pragma unroll
        for (int j = 0; j < DTILES; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
        m_run[0] = m_run[1] = -INFINITY;
        l_run[0] = l_run[1] = 0.f;
    };

    // Write the segment's result: final output if the segment is the whole
    // pair, else a partial in slot (pair index + c).
    auto end_segment = [&](bool whole_pair) {
        // full row sums of this warp
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            l_run[r] += __shfl_xor_sync(kFull, l_run[r], 1);
            l_run[r] += __shfl_xor_sync(kFull, l_run[r], 2);
        }
        const int pair = w.b * p.Hkv + w.h;
        const size_t slot = (size_t)pair + c;
        float f[2], lse2[2];  // factor applied to this warp's O; row lse in log2 units
        if (ks == 1) {
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                f[r] = l_run[r] > 0.f ? 1.f / l_run[r] : 0.f;
                lse2[r] = l_run[r] > 0.f ? m_run[r] + __log2f(l_run[r]) : -INFINITY;
            }
        } else {
            named_bar_sync(1, 32 * kConsumerWarps);
            for (int i = threadIdx.x; i < mt_pad * 16 * D; i += 32 * kConsumerWarps) epi[i] = 0.f;
            if ((lane & 3) == 0) {
                xml[(warp * 16 + quad_row) * 2 + 0] = m_run[0];
                xml[(warp * 16 + quad_row) * 2 + 1] = l_run[0];
                xml[(warp * 16 + quad_row + 8) * 2 + 0] = m_run[1];
                xml[(warp * 16 + quad_row + 8) * 2 + 1] = l_run[1];
            }
            named_bar_sync(1, 32 * kConsumerWarps);
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int rr = quad_row + 8 * r;
                float M = -INFINITY;
                for (int k2 = 0; k2 < ks; ++k2) M = fmaxf(M, xml[((mw + k2 * mt_pad) * 16 + rr) * 2]);
                const float Mu = M == -INFINITY ? 0.f : M;
                float L = 0.f;
                for (int k2 = 0; k2 < ks; ++k2) {
                    const int ww = mw + k2 * mt_pad;
                    L += ex2(xml[(ww * 16 + rr) * 2] - Mu) * xml[(ww * 16 + rr) * 2 + 1];
                }
                f[r] = L > 0.f ? ex2(m_run[r] - Mu) / L : 0.f;
                lse2[r] = L > 0.f ? Mu + __log2f(L) : -INFINITY;
            }
            float *er = epi + (size_t)mw * 16 * D;
#pragma unroll
            for (int j = 0; j < DTILES; ++j) {
                const int col = j * 8 + quad_col;
                atomicAdd(er + quad_row * D + col, o[j][0] * f[0]);
                atomicAdd(er + quad_row * D + col + 1, o[j][1] * f[0]);
                atomicAdd(er + (quad_row + 8) * D + col, o[j][2] * f[1]);
                atomicAdd(er + (quad_row + 8) * D + col + 1, o[j][3] * f[1]);
            }
            named_bar_sync(1, 32 * kConsumerWarps);
        }

        // Rows of this warp's m-tile; with ks > 1 warp kw == 0 writes them
        // from shared memory, with ks == 1 every warp writes from registers.
        if (ks == 1 || kw == 0) {
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int row = r == 0 ? rowA : rowB;
                if (row >= rows_active) continue;
                const int i = row / p.G, g = row % p.G;
                float v[DTILES][2];
#pragma unroll
                for (int j = 0; j < DTILES; ++j) {
                    const int col = j * 8 + quad_col;
                    if (ks == 1) {
                        v[j][0] = o[j][2 * r] * f[r];
                        v[j][1] = o[j][2 * r + 1] * f[r];
                    } else {
                        const float *er = epi + ((size_t)mw * 16 + quad_row + 8 * r) * D;
                        v[j][0] = er[col];
                        v[j][1] = er[col + 1];
                    }
                }
                if (whole_pair) {
                    uint16_t *orow = p.out + (((size_t)w.b * p.max_block + i) * p.Hq +
                                              (size_t)w.h * p.G + g) * D;
#pragma unroll
                    for (int j = 0; j < DTILES; ++j)
                        *reinterpret_cast<uint32_t *>(orow + j * 8 + quad_col) =
                            pack_bf16(v[j][0], v[j][1]);
                    if ((lane & 3) == 0)
                        p.lse[((size_t)w.b * p.Hq + (size_t)w.h * p.G + g) * p.max_block + i] =
                            lse2[r] * kLn2;
                } else {
                    float *prow = p.part_o + (slot * p.rows_max + row) * D;
#pragma unroll
                    for (int j = 0; j < DTILES; ++j)
                        *reinterpret_cast<float2 *>(prow + j * 8 + quad_col) =
                            make_float2(v[j][0], v[j][1]);
                    if ((lane & 3) == 0) p.part_lse[slot * p.rows_max + row] = lse2[r] * kLn2;
                }
            }
        }
        // Whole pair written here: rows past the block are 0 with lse -inf.
        if (whole_pair) {
            const int nthr = 32 * kConsumerWarps;
            for (int idx = threadIdx.x; idx < (p.rows_max - rows_active) * (D / 2); idx += nthr) {
                const int row = rows_active + idx / (D / 2), col = (idx % (D / 2)) * 2;
                const int i = row / p.G, g = row % p.G;
                *reinterpret_cast<uint32_t *>(p.out + (((size_t)w.b * p.max_block + i) * p.Hq +
                                                       (size_t)w.h * p.G + g) * D + col) = 0u;
                if (col == 0)
                    p.lse[((size_t)w.b * p.Hq + (size_t)w.h * p.G + g) * p.max_block + i] =
                        -INFINITY;
            }
        }
    };

    begin_segment(lo);
    for (long long g = lo, k = 0; g < hi; ++g, ++k) {
        const int s = (int)(k % STAGES);
        const uint32_t ph = (uint32_t)((k / STAGES) & 1);
        const bool ok = __all_sync(kFull, mbar_wait(full0 + 8 * s, ph, abort_flag, p.status));
        const bool block_tile = (w.t == w.nt - 1);
        // keys of this tile that exist: prefix positions < P, block rows < T
        const int nvalid = block_tile ? w.T : min(kTileKeys, w.P - w.t * kTileKeys);
        const uint32_t kt = smem_u32(stage_base + s * S::kStageBytes);
        const uint32_t vt = kt + S::kTileBytes;
        const int key0 = kw * kpw;  // first key of this warp inside the tile
        const int nt8 = kpw / 8;    // n-tiles of 8 keys handled by this warp
        if (ok && mw * 16 < rows_active) {
            // ---- S = Q K^T over this warp's keys ----
            float sc[8][4];
#pragma unroll
            for (int j = 0; j < 8; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < KSTEPS; ++kk) {
#pragma unroll
                for (int jp = 0; jp < 4; ++jp) {
                    if (jp * 2 < nt8) {
                        const int key = key0 + jp * 16 + (lane & 7) + ((lane >> 4) << 3);
                        const int cg = 2 * kk + ((lane >> 3) & 1);
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(swz(kt, key, cg), b0, b1, b2, b3);
                        mma_bf16(sc[2 * jp], qa[kk], b0, b1);
                        mma_bf16(sc[2 * jp + 1], qa[kk], b2, b3);
                    }
                }
            }
            // ---- mask, scale, online softmax (base 2) ----
            float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (j < nt8) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int key = key0 + j * 8 + quad_col + (e & 1);
                        const int r = e >> 1;
                        bool valid = key < nvalid;
                        if (block_tile) valid = valid && key <= (r ? iB : iA);
                        const float x = valid ? sc[j][e] * p.scale_log2 : -INFINITY;
                        sc[j][e] = x;
                        tmax[r] = fmaxf(tmax[r], x);
                    }
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
            // P = 2^(s - m), kept in place of the scores
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (j < nt8) {
                    sc[j][0] = ex2(sc[j][0] - mu[0]);
                    sc[j][1] = ex2(sc[j][1] - mu[0]);
                    sc[j][2] = ex2(sc[j][2] - mu[1]);
                    sc[j][3] = ex2(sc[j][3] - mu[1]);
                    l_run[0] += sc[j][0] + sc[j][1];
                    l_run[1] += sc[j][2] + sc[j][3];
                }
            }
            // ---- O += P V ----
            const bool tail = nvalid < key0 + kpw;
#pragma unroll
            for (int kk2 = 0; kk2 < 4; ++kk2) {
                if (kk2 * 16 < kpw) {
                    const int kb = key0 + kk2 * 16;
                    // P of keys kb..kb+15 as the A fragment of m16n8k16
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
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty0 + 8 * s);
        if (threadIdx.x == 0 && pg < hi) issue_next();

        // segment ends at the pair's last tile or at the end of the range
        if (block_tile || g + 1 == hi) {
            const bool whole = (seg_first == pair_first) && block_tile;
            end_segment(whole);
            walk_next(p, w);
            if (g + 1 < hi) begin_segment(g + 1);
        } else {
            walk_next(p, w);
        }
    }
}

// Merge the partials of every pair that more than one CTA worked on.
template <int D>
__global__ void __launch_bounds__(256) merge_kernel(const AttnParams p) {
    const int pair = blockIdx.x;
    const int b = pair / p.Hkv, h = pair % p.Hkv;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __shared__ long long s_first, s_N;
    if (warp == 0) {
        const long long N = total_tiles(p);
        long long before = 0;
        for (int bb = lane; bb < b; bb += 32) before += (long long)tiles_of(clamp_prefix(p, bb)) * p.Hkv;
#pragma unroll
        for (int d = 16; d > 0; d >>= 1) before += __shfl_xor_sync(kFull, before, d);
        if (lane == 0) {
            s_N = N;
            s_first = before + (long long)h * tiles_of(clamp_prefix(p, b));
        }
    }
    __syncthreads();
    const long long N = s_N, first = s_first;
    const long long last = first + tiles_of(clamp_prefix(p, b)) - 1;
    const int c0 = cta_of(first, N, p.num_ctas), c1 = cta_of(last, N, p.num_ctas);
    // CTAs with an empty range (more CTAs than tiles) hold no partial
    const int C = p.num_ctas;
    auto nonempty = [&](int cc) {
        return (long long)cc * N / C != (long long)(cc + 1) * N / C;
    };
    int nseg = 0;
    for (int cc = c0; cc <= c1; ++cc) nseg += nonempty(cc);
    if (nseg <= 1) return;  // the single CTA wrote the final result itself
    const int T = clamp_block(p, b);
    const int rows_active = p.G * T;
    constexpr int VPL = D / 32;  // values per lane
    for (int row = warp; row < p.rows_max; row += 8) {
        const int i = row / p.G, g = row % p.G;
        uint16_t *orow = p.out + (((size_t)b * p.max_block + i) * p.Hq + (size_t)h * p.G + g) * D;
        float *lrow = p.lse + ((size_t)b * p.Hq + (size_t)h * p.G + g) * p.max_block + i;
        if (row >= rows_active) {
            for (int d = lane; d < D; d += 32) orow[d] = 0;
            if (lane == 0) *lrow = -INFINITY;
            continue;
        }
        float M = -INFINITY;
        for (int cc = c0; cc <= c1; ++cc)
            if (nonempty(cc)) M = fmaxf(M, p.part_lse[((size_t)pair + cc) * p.rows_max + row]);
        float L = 0.f, acc[VPL];
#pragma unroll
        for (int v = 0; v < VPL; ++v) acc[v] = 0.f;
        for (int cc = c0; cc <= c1; ++cc) {
            if (!nonempty(cc)) continue;
            const size_t slot = (size_t)pair + cc;
            const float wgt = __expf(p.part_lse[slot * p.rows_max + row] - M);
            L += wgt;
            const float *prow = p.part_o + (slot * p.rows_max + row) * D + lane * VPL;
            if constexpr (VPL == 4) {
                const float4 x = *reinterpret_cast<const float4 *>(prow);
                acc[0] += wgt * x.x;
                acc[1] += wgt * x.y;
                acc[2] += wgt * x.z;
                acc[3] += wgt * x.w;
            } else {
                const float2 x = *reinterpret_cast<const float2 *>(prow);
                acc[0] += wgt * x.x;
                acc[1] += wgt * x.y;
            }
        }
        const float inv = 1.f / L;
        if constexpr (VPL == 4) {
            uint2 pk;
            pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
            pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
            *reinterpret_cast<uint2 *>(orow + lane * VPL) = pk;
        } else {
            *reinterpret_cast<uint32_t *>(orow + lane * VPL) = pack_bf16(acc[0] * inv, acc[1] * inv);
        }
        if (lane == 0) *lrow = M + __logf(L);
    }
}

template <int D>
constexpr int kStages = (D == 128) ? 2 : 4;

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
    attn_kernel<D, ST><<<p.num_ctas, kAttnThreads, smem, stream>>>(tk, tv, tkb, tvb, p);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    merge_kernel<D><<<p.B * p.Hkv, 256, 0, stream>>>(p);
    return cudaGetLastError();
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

cudaError_t attn_launch(const AttnParams &p, int head_dim, const CUtensorMap &tm_k,
                        const CUtensorMap &tm_v, const CUtensorMap &tm_kb,
                        const CUtensorMap &tm_vb, cudaStream_t stream) {
    if (head_dim == 128) return launch_d<128>(p, tm_k, tm_v, tm_kb, tm_vb, stream);
    if (head_dim == 64) return launch_d<64>(p, tm_k, tm_v, tm_kb, tm_vb, stream);
    return cudaErrorInvalidValue;
}

}  // namespace das
