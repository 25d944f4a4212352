// das_commit.cu -- greedy acceptance and the multi-depth cache commit
// (Sec. 3.4; App. B.1) on sm_103a.
//
// Every kernel here is launched as a programmatic dependent of the previous
// kernel in the stream: it reads nothing before griddepcontrol.wait, and
// every CTA executes that wait.
#include <atomic>

#include <cooperative_groups.h>

#include "das_internal.h"

namespace cg = cooperative_groups;

namespace das {
namespace {

// ---- greedy acceptance and the DAS-Wave readout ------------------------------
// No scratch memory beyond the outputs.  Greedy acceptance takes one of two
// forms, chosen per launch:
//   accept_fused_kernel (one kernel): a cluster of W * k CTAs is one
//     sequence, row i scanned by CTAs i k .. i k + k - 1 (each a 1/k slice
//     of the vocabulary); every CTA stores its best (value, index) straight
//     into CTA 0's shared memory (distributed shared memory), and CTA 0
//     writes target_ids[b][*], accepted[b] and next_token[b].  Used when
//     W k <= 16 (k reduced to fit) and all B clusters are resident at once.
//   row_argmax_kernel + accept_scan_kernel (two kernels): a cluster of k
//     CTAs is one row, CTA 0 writes target_ids[b][i]; then one warp per
//     sequence (a programmatic dependent) finds the first mismatch between
//     draft_ids and target_ids and writes accepted and next_token.  It
//     spreads rows over more SMs, and serves any B and W.
// k is chosen so that rows * k fills the SMs (at most 8).  The DAS-Wave
// readout (Eq. 6, Sec. 3.3) is row_argmax_kernel in readout mode, writing
// tokens[b][i + 1].
constexpr int kRowThreadsMax = 1024;
constexpr int kRowLoads = 8;    // vector loads in flight per thread
constexpr int kMaxRowCtas = 8;  // CTAs per row: a portable cluster
constexpr int kMaxSeqCtas = 16; // CTAs of one sequence's cluster (a non-portable size)
constexpr int kMaxW = 1024;
constexpr int kScanWarps = 4;

// (value, index) order of the argmax: larger value wins, equal values go to
// the smaller index, so the result is the first maximum.
__device__ __forceinline__ void better(float &bv, int &bi, float v, int i) {
    if (v > bv || (v == bv && i < bi)) {
        bv = v;
        bi = i;
    }
}
__device__ __forceinline__ void warp_best(float &bv, int &bi) {
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, d);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, d);
        better(bv, bi, ov, oi);
    }
}

struct RowArgs {
    const float *logits;  // [B][W][vocab]
    int W, vocab, slice;  // slice: floats per CTA, a multiple of the vector width
    int32_t *target_ids;  // accept mode: [B][W]
    int32_t *tokens;      // readout mode: [B][stride]
    int stride;
};

// The first maximum (value, index) of logits src[lo, hi) over the whole CTA
// (valid in thread 0): batches of kRowLoads vector loads per thread, all
// issued before the compares, then warp and CTA reductions.  VEC = 4: float4
// loads (vocab % 4 == 0 and 16-byte aligned logits, lo a multiple of 4), else 1.
template <int VEC>
__device__ __forceinline__ void slice_best(const float *__restrict__ row, int lo, int hi,
                                           float &bv, int &bi, float *warp_v, int *warp_i) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nvec = (hi - lo) / VEC;  // the slice is a multiple of VEC
    const float *__restrict__ src = row + lo;
    bv = -INFINITY;
    bi = 0x7fffffff;
    const int nt = blockDim.x;
    for (int j0 = threadIdx.x; j0 < nvec; j0 += kRowLoads * nt) {
        float x[kRowLoads][VEC];
#pragma unroll
        for (int u = 0; u < kRowLoads; ++u) {
            const int j = j0 + u * nt;
            if (j < nvec) {
                if (VEC == 4) {
                    const float4 y = __ldcs(reinterpret_cast<const float4 *>(src) + j);
                    x[u][0] = y.x;
                    x[u][1 % VEC] = y.y;
                    x[u][2 % VEC] = y.z;
                    x[u][VEC - 1] = y.w;
                } else {
                    x[u][0] = __ldcs(src + j);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kRowLoads; ++u) {
            const int j = j0 + u * nt;
            if (j < nvec) {
#pragma unroll
                for (int e = 0; e < VEC; ++e) better(bv, bi, x[u][e], lo + VEC * j + e);
            }
        }
    }
    warp_best(bv, bi);
    if (lane == 0) {
        warp_v[warp] = bv;
        warp_i[warp] = bi;
    }
    __syncthreads();
    if (warp == 0) {
        bv = lane < (nt >> 5) ? warp_v[lane] : -INFINITY;
        bi = lane < (nt >> 5) ? warp_i[lane] : 0x7fffffff;
        warp_best(bv, bi);
    }
}

// The cluster size k (1..8) is the launch's; row = blockIdx.x / k.
template <int VEC, bool READOUT>
__global__ void __launch_bounds__(kRowThreadsMax) row_argmax_kernel(const RowArgs a) {
    __shared__ float warp_v[32];
    __shared__ int warp_i[32];
    __shared__ float cand_v[kMaxRowCtas];
    __shared__ int cand_i[kMaxRowCtas];
    cg::cluster_group cluster = cg::this_cluster();
    const int k = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const size_t row = blockIdx.x / k;
    // a CTA's shared memory may be written by another only once that CTA has
    // started: every CTA arrives here and waits before its remote store
    if (k > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // the logits may come from the kernel before this one
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const int lo = min(rank * a.slice, a.vocab), hi = min(lo + a.slice, a.vocab);
    float bv;
    int bi;
    slice_best<VEC>(a.logits + row * (size_t)a.vocab, lo, hi, bv, bi, warp_v, warp_i);
    if (k > 1) {
        asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
        if (threadIdx.x == 0) {
            *cluster.map_shared_rank(cand_v + rank, 0) = bv;
            *cluster.map_shared_rank(cand_i + rank, 0) = bi;
        }
        // the candidates are in CTA 0 once every CTA has arrived (release);
        // only CTA 0 waits, and only its shared memory is read remotely
        asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
        if (rank != 0) return;
        asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
        if (threadIdx.x == 0) {
            bv = cand_v[0];
            bi = cand_i[0];
            for (int r = 1; r < k; ++r) better(bv, bi, cand_v[r], cand_i[r]);
        }
    }
    if (threadIdx.x == 0) {
        // a row of -inf keeps the sentinel: the first index wins
        const int t = bi == 0x7fffffff ? 0 : bi;
        if (READOUT) {
            const size_t b = row / a.W, i = row % a.W;
            a.tokens[b * a.stride + i + 1] = t;
        } else {
            a.target_ids[row] = t;
        }
    }
}

// Greedy acceptance in one kernel.  The launch's cluster of n = W k CTAs
// (n <= 16) is sequence b = blockIdx.x / n; CTA rank i k + r scans slice r
// of row i.  CTA 0 gathers the n candidates, and its first warp (lane i for
// row i) writes target_ids[b][i], then accepted[b] (the first mismatch with
// draft_ids, by ballot) and next_token[b].
template <int VEC>
__global__ void __launch_bounds__(kRowThreadsMax)
    accept_fused_kernel(const RowArgs a, const int32_t *__restrict__ draft,
                        int32_t *__restrict__ accepted, int32_t *__restrict__ next_token) {
    __shared__ float warp_v[32];
    __shared__ int warp_i[32];
    __shared__ float cand_v[kMaxSeqCtas];
    __shared__ int cand_i[kMaxSeqCtas];
    cg::cluster_group cluster = cg::this_cluster();
    const int n = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int k = n / a.W;
    const size_t b = blockIdx.x / n;
    const int i = rank / k, r = rank % k;
    if (n > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // the logits and draft ids may come from the kernel before this one
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const int lo = min(r * a.slice, a.vocab), hi = min(lo + a.slice, a.vocab);
    float bv;
    int bi;
    slice_best<VEC>(a.logits + (b * a.W + i) * (size_t)a.vocab, lo, hi, bv, bi, warp_v, warp_i);
    if (n > 1) {
        asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
        if (threadIdx.x == 0) {
            *cluster.map_shared_rank(cand_v + rank, 0) = bv;
            *cluster.map_shared_rank(cand_i + rank, 0) = bi;
        }
        // as in row_argmax_kernel: only CTA 0 waits and is read remotely
        asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
        if (rank != 0) return;
        asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
    } else if (threadIdx.x == 0) {
        cand_v[0] = bv;
        cand_i[0] = bi;
    }
    if (n == 1) __syncthreads();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        const int32_t *d = draft + b * a.W;
        int t = 0;
        bool miss = false;
        if (lane < a.W) {
            float v = cand_v[lane * k];
            int x = cand_i[lane * k];
            for (int u = 1; u < k; ++u) better(v, x, cand_v[lane * k + u], cand_i[lane * k + u]);
            t = x == 0x7fffffff ? 0 : x;  // a row of -inf: the first index
            a.target_ids[b * a.W + lane] = t;
            miss = d[lane] != t;
        }
        const unsigned m = __ballot_sync(0xffffffffu, miss);
        const int first = m ? __ffs(m) - 1 : a.W;
        const int t_first = __shfl_sync(0xffffffffu, t, first < a.W ? first : 0);
        if (lane == 0) {
            accepted[b] = first;
            next_token[b] = first < a.W ? t_first : d[a.W - 1];
        }
    }
}

// accepted[b] = first i with draft[b][i] != target_ids[b][i] (W if none);
// next_token[b] = target_ids[b][accepted[b]], or draft[b][W - 1] if all W
// proposals were accepted.  One warp per sequence.
__global__ void __launch_bounds__(kScanWarps * 32)
    accept_scan_kernel(const int32_t *__restrict__ target_ids, const int32_t *__restrict__ draft,
                       int B, int W, int32_t *__restrict__ accepted,
                       int32_t *__restrict__ next_token) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int lane = threadIdx.x & 31;
    const long long b = (long long)blockIdx.x * kScanWarps + (threadIdx.x >> 5);
    if (b >= B) return;
    const int32_t *t = target_ids + b * W, *d = draft + b * W;
    int first = W;
    for (int i0 = 0; i0 < W; i0 += 32) {
        const int i = i0 + lane;
        const unsigned m = __ballot_sync(0xffffffffu, i < W && d[i] != t[i]);
        if (m) {
            first = i0 + __ffs(m) - 1;
            break;
        }
    }
    if (lane == 0) {
        accepted[b] = first;
        next_token[b] = first < W ? t[first] : d[W - 1];
    }
}

// ---- commit ---------------------------------------------------------------------
constexpr int kCopyThreads = 256;
constexpr int kCopyUnroll = 4;
constexpr int kCopyChunk = kCopyThreads * kCopyUnroll;  // 16-byte words per CTA and tensor

__device__ __forceinline__ int append_count(int32_t a, int W) {
    if (a < 0) a = 0;
    return a + 1 < W ? a + 1 : W;
}

// Copy of the materialized inputs' K/V.  CTA x handles chunk x % chunks of
// slab x / chunks, slab = (depth * layers + layer) * batch + b; each thread
// moves kCopyUnroll 16-byte words of K and of V, all loads before the stores.
__global__ void __launch_bounds__(kCopyThreads)
    append_copy_kernel(uint4 *__restrict__ kc, uint4 *__restrict__ vc,
                       const uint4 *__restrict__ kn, const uint4 *__restrict__ vn,
                       const int32_t *__restrict__ accepted,
                       const int32_t *__restrict__ prefix_len, int batch, int capacity, int W,
                       int row_words, int chunks) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const size_t slab = blockIdx.x / chunks;
    const int chunk = blockIdx.x % chunks;
    const int b = (int)(slab % batch);
    const int n = append_count(accepted[b], W);
    const int p = prefix_len[b];
    if (p < 0 || p + n > capacity) return;  // reported by append_finalize_kernel
    const int words = n * row_words;
    const int w0 = chunk * kCopyChunk + threadIdx.x;
    if (chunk * kCopyChunk >= words) return;
    const uint4 *ks = kn + slab * W * row_words;
    const uint4 *vs = vn + slab * W * row_words;
    uint4 *kd = kc + (slab * capacity + p) * row_words;
    uint4 *vd = vc + (slab * capacity + p) * row_words;
    uint4 a[kCopyUnroll], c[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
        const int w = w0 + u * kCopyThreads;
        if (w < words) {
            a[u] = __ldcs(ks + w);
            c[u] = __ldcs(vs + w);
        }
    }
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
        const int w = w0 + u * kCopyThreads;
        if (w < words) {
            kd[w] = a[u];
            vd[w] = c[u];
        }
    }
}

// Two bf16 (element 0 in the low half) -> two e4m3 (element 0 in bits 0-7):
// round to nearest, ties to even; beyond +-448 (and +-inf) saturate to +-448.
__device__ __forceinline__ uint32_t bf16x2_to_e4m3x2(uint32_t w) {
    const float lo = __uint_as_float(w << 16), hi = __uint_as_float(w & 0xffff0000u);
    uint32_t r;
    asm("{\n .reg .b16 t;\n cvt.rn.satfinite.e4m3x2.f32 t, %1, %2;\n cvt.u32.u16 %0, t;\n}"
        : "=r"(r)
        : "f"(hi), "f"(lo));
    return r;
}

// das_kv_append_f8: as append_copy_kernel, over the staged [R][L][B][W][Hkv][D]
// K/V; slabs of depth R are copied to the bf16 top tensors, slabs of lower
// depths rounded to e4m3 (8 bytes per 16-byte bf16 word) into the low ones.
__global__ void __launch_bounds__(kCopyThreads)
    append_f8_kernel(uint4 *__restrict__ k_top, uint4 *__restrict__ v_top,
                     uint2 *__restrict__ k_low, uint2 *__restrict__ v_low,
                     const uint4 *__restrict__ kn, const uint4 *__restrict__ vn,
                     const int32_t *__restrict__ accepted, const int32_t *__restrict__ prefix_len,
                     int depths, int layers, int batch, int capacity, int W, int row_words,
                     int chunks) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const size_t slab = blockIdx.x / chunks;
    const int chunk = blockIdx.x % chunks;
    const int b = (int)(slab % batch);
    const int dl = (int)(slab / batch), d = dl / layers, l = dl % layers;
    const int n = append_count(accepted[b], W);
    const int p = prefix_len[b];
    if (p < 0 || p + n > capacity) return;  // reported by append_finalize_kernel
    const int words = n * row_words;
    const int w0 = chunk * kCopyChunk + threadIdx.x;
    if (chunk * kCopyChunk >= words) return;
    const uint4 *ks = kn + slab * W * row_words;
    const uint4 *vs = vn + slab * W * row_words;
    uint4 a[kCopyUnroll], c[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
        const int w = w0 + u * kCopyThreads;
        if (w < words) {
            a[u] = __ldcs(ks + w);
            c[u] = __ldcs(vs + w);
        }
    }
    if (d == depths - 1) {
        const size_t o = (((size_t)l * batch + b) * capacity + p) * row_words;
#pragma unroll
        for (int u = 0; u < kCopyUnroll; ++u) {
            const int w = w0 + u * kCopyThreads;
            if (w < words) {
                k_top[o + w] = a[u];
                v_top[o + w] = c[u];
            }
        }
    } else {
        const size_t o = ((((size_t)d * layers + l) * batch + b) * capacity + p) * row_words;
        auto q8 = [](uint4 x) {
            return make_uint2(bf16x2_to_e4m3x2(x.x) | bf16x2_to_e4m3x2(x.y) << 16,
                              bf16x2_to_e4m3x2(x.z) | bf16x2_to_e4m3x2(x.w) << 16);
        };
#pragma unroll
        for (int u = 0; u < kCopyUnroll; ++u) {
            const int w = w0 + u * kCopyThreads;
            if (w < words) {
                k_low[o + w] = q8(a[u]);
                v_low[o + w] = q8(c[u]);
            }
        }
    }
}

// Runs once every copy has read prefix_len: grow it or flag the sequence.
__global__ void append_finalize_kernel(const int32_t *__restrict__ accepted,
                                       int32_t *__restrict__ prefix_len, int batch, int capacity,
                                       int W, int32_t *__restrict__ error_flag) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < batch; b += gridDim.x * blockDim.x) {
        const int n = append_count(accepted[b], W);
        const int p = prefix_len[b];
        if (p < 0 || p + n > capacity) {
            *error_flag = 1;
        } else {
            prefix_len[b] = p + n;
        }
    }
}

template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, unsigned cluster,
                       cudaStream_t stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    int n = 1;
    if (cluster > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = cluster;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        n = 2;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Params>(args)...);
}

// CTAs per row of the argmax step: k = SMs / rows clamped to [1, 8].
int row_ctas(long long rows, int sms) {
    return rows >= sms ? 1 : (int)std::min<long long>(kMaxRowCtas, sms / rows);
}

// Threads of an argmax CTA: enough for kRowLoads vector loads each over the
// slice (a.slice must be set), a multiple of 32 in [32, 1024].
template <int VEC>
int row_threads(const RowArgs &a) {
    const int nvec = a.slice / VEC;
    const int t = (nvec + kRowLoads - 1) / kRowLoads;
    return std::max(32, std::min(kRowThreadsMax, (t + 31) / 32 * 32));
}

// The argmax step: k CTAs per row, k = SMs / rows clamped to [1, 8], with
// enough threads for kRowLoads vector loads each over a 1/k slice.
template <int VEC, bool READOUT>
cudaError_t row_argmax_launch(RowArgs a, long long rows, cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int sms = attn_grid_size(dev);
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int k = row_ctas(rows, sms);
    const int slice = (a.vocab + k - 1) / k;
    a.slice = (slice + VEC - 1) / VEC * VEC;
    if (rows * k > 0x7fffffffLL) return cudaErrorInvalidValue;
    return launch_pdl(row_argmax_kernel<VEC, READOUT>, dim3((unsigned)(rows * k)),
                      dim3((unsigned)row_threads<VEC>(a)), (unsigned)k, stream, a);
}

cudaError_t argmax_launch(const RowArgs &a, int B, bool readout, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if (a.W < 1 || a.W > kMaxW) return cudaErrorInvalidValue;
    const long long rows = (long long)B * a.W;
    const bool vec = (a.vocab % 4) == 0 && (reinterpret_cast<uintptr_t>(a.logits) & 15u) == 0;
    if (readout)
        return vec ? row_argmax_launch<4, true>(a, rows, stream)
                   : row_argmax_launch<1, true>(a, rows, stream);
    return vec ? row_argmax_launch<4, false>(a, rows, stream)
               : row_argmax_launch<1, false>(a, rows, stream);
}

// Clusters of n CTAs of kRowThreadsMax threads (an upper bound on the
// launch's) that can be resident at once, looked up once per device and n.
template <int VEC>
cudaError_t fused_resident_clusters(int dev, int n, int &clusters) {
    static std::atomic<int> cached[64][kMaxSeqCtas + 1];
    if (dev < 64) {
        const int c = cached[dev][n].load(std::memory_order_relaxed);
        if (c > 0) {
            clusters = c - 1;
            return cudaSuccess;
        }
    }
    cudaError_t e = cudaFuncSetAttribute(accept_fused_kernel<VEC>,
                                         cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)n);
    cfg.blockDim = dim3(kRowThreadsMax);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)n;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaOccupancyMaxActiveClusters(&clusters, accept_fused_kernel<VEC>, &cfg);
    if (e != cudaSuccess) return e;
    if (dev < 64) cached[dev][n].store(clusters + 1, std::memory_order_relaxed);
    return cudaSuccess;
}

// k > 0: greedy acceptance runs as accept_fused_kernel with k CTAs per row
// (the two-kernel form's k, or fewer so that W k <= 16) when every
// sequence's cluster of W k CTAs is resident at once (one wave); otherwise
// k = 0 (the two-kernel form).  On a 152-SM GB300 at most 7 clusters of 16
// CTAs (15 of 8) are resident, so [8, 16, vocab] stays two-kernel, while a
// single sequence's accept (B 1, W 8) gains the second kernel's dependency
// wait: 6.18 -> 5.02 us over a 32000 vocabulary (B 2 to 4 at W 16: equal).
cudaError_t fused_accept_ctas(int B, int W, bool vec, int &k) {
    k = 0;
    if (W > kMaxSeqCtas) return cudaSuccess;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int sms = attn_grid_size(dev);
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int kr = std::min(row_ctas((long long)B * W, sms), kMaxSeqCtas / W);
    int clusters = 0;
    e = vec ? fused_resident_clusters<4>(dev, W * kr, clusters)
            : fused_resident_clusters<1>(dev, W * kr, clusters);
    if (e != cudaSuccess) {  // a device without that cluster size: the two-kernel form
        (void)cudaGetLastError();
        return cudaSuccess;
    }
    if (B <= clusters) k = kr;
    return cudaSuccess;
}

template <int VEC>
cudaError_t accept_fused_launch(RowArgs a, int B, int k, const int32_t *draft,
                                int32_t *accepted, int32_t *next_token, cudaStream_t stream) {
    const int slice = (a.vocab + k - 1) / k;
    a.slice = (slice + VEC - 1) / VEC * VEC;
    const int n = a.W * k;
    return launch_pdl(accept_fused_kernel<VEC>, dim3((unsigned)(B * n)),
                      dim3((unsigned)row_threads<VEC>(a)), (unsigned)n, stream, a, draft,
                      accepted, next_token);
}

}  // namespace

cudaError_t accept_launch(const float *logits, const int32_t *draft, int B, int W, int vocab,
                          int32_t *accepted, int32_t *target_ids, int32_t *next_token,
                          cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    RowArgs a = {};
    a.logits = logits;
    a.W = W;
    a.vocab = vocab;
    a.target_ids = target_ids;
    const bool vec = (vocab % 4) == 0 && (reinterpret_cast<uintptr_t>(logits) & 15u) == 0;
    int k = 0;
    cudaError_t e = fused_accept_ctas(B, W, vec, k);
    if (e != cudaSuccess) return e;
    if (k > 0)
        return vec ? accept_fused_launch<4>(a, B, k, draft, accepted, next_token, stream)
                   : accept_fused_launch<1>(a, B, k, draft, accepted, next_token, stream);
    e = argmax_launch(a, B, false, stream);
    if (e != cudaSuccess) return e;
    return launch_pdl(accept_scan_kernel, dim3((unsigned)((B + kScanWarps - 1) / kScanWarps)),
                      dim3(kScanWarps * 32), 1, stream, static_cast<const int32_t *>(target_ids),
                      draft, B, W, accepted, next_token);
}

cudaError_t wave_readout_launch(const float *logits, int B, int W, int vocab, int32_t *tokens,
                                int stride, cudaStream_t stream) {
    RowArgs a = {};
    a.logits = logits;
    a.W = W;
    a.vocab = vocab;
    a.tokens = tokens;
    a.stride = stride;
    return argmax_launch(a, B, true, stream);
}

cudaError_t append_launch(const das_kv_cache &c, const void *k_new, const void *v_new,
                          const int32_t *accepted, int W, int32_t *prefix_len,
                          int32_t *error_flag, cudaStream_t stream) {
    const int row_words = c.kv_heads * c.head_dim * 2 / 16;
    const long long slabs = (long long)c.depths * c.layers * c.batch;
    if (slabs == 0) return cudaSuccess;
    const long long words = (long long)W * row_words;
    if (words > 0x7fffffffLL) return cudaErrorInvalidValue;
    const int chunks = (int)((words + kCopyChunk - 1) / kCopyChunk);
    if (slabs * chunks > 0x7fffffffLL) return cudaErrorInvalidValue;
    cudaError_t e = launch_pdl(append_copy_kernel, dim3((unsigned)(slabs * chunks)),
                               dim3(kCopyThreads), 1, stream, static_cast<uint4 *>(c.k),
                               static_cast<uint4 *>(c.v), static_cast<const uint4 *>(k_new),
                               static_cast<const uint4 *>(v_new), accepted,
                               static_cast<const int32_t *>(prefix_len), c.batch, c.capacity, W,
                               row_words, chunks);
    if (e != cudaSuccess) return e;
    return launch_pdl(append_finalize_kernel, dim3((unsigned)((c.batch + 127) / 128)), dim3(128),
                      1, stream, accepted, prefix_len, c.batch, c.capacity, W, error_flag);
}

cudaError_t append_f8_launch(const das_kv_cache_f8 &c, const void *k_new, const void *v_new,
                             const int32_t *accepted, int W, int32_t *prefix_len,
                             int32_t *error_flag, cudaStream_t stream) {
    const int row_words = c.kv_heads * c.head_dim * 2 / 16;
    const long long slabs = (long long)c.depths * c.layers * c.batch;
    const long long words = (long long)W * row_words;
    if (words > 0x7fffffffLL) return cudaErrorInvalidValue;
    const int chunks = (int)((words + kCopyChunk - 1) / kCopyChunk);
    if (slabs * chunks > 0x7fffffffLL) return cudaErrorInvalidValue;
    cudaError_t e = launch_pdl(
        append_f8_kernel, dim3((unsigned)(slabs * chunks)), dim3(kCopyThreads), 1, stream,
        static_cast<uint4 *>(c.k_top), static_cast<uint4 *>(c.v_top),
        static_cast<uint2 *>(c.k_low), static_cast<uint2 *>(c.v_low),
        static_cast<const uint4 *>(k_new), static_cast<const uint4 *>(v_new), accepted,
        static_cast<const int32_t *>(prefix_len), c.depths, c.layers, c.batch, c.capacity, W,
        row_words, chunks);
    if (e != cudaSuccess) return e;
    return launch_pdl(append_finalize_kernel, dim3((unsigned)((c.batch + 127) / 128)), dim3(128),
                      1, stream, accepted, prefix_len, c.batch, c.capacity, W, error_flag);
}

}  // namespace das
