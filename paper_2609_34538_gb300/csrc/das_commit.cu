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
// Two steps, neither with scratch memory beyond the outputs:
//   row_argmax_kernel: the first maximum of every logits row, row i of
//     sequence b scanned by k CTAs (a cluster of k, each a 1/k slice of the
//     vocabulary, k chosen so that rows * k fills the SMs, at most 8); CTA r
//     of the cluster stores its best (value, index) straight into CTA 0's
//     shared memory (distributed shared memory) and CTA 0 writes
//       accept mode (Sec. 3.4):  target_ids[b][i];
//       readout mode (Eq. 6, Sec. 3.3):  tokens[b][i + 1];
//   accept_scan_kernel (accept mode only, a programmatic dependent of the
//     first): one warp per sequence finds the first mismatch between
//     draft_ids and target_ids and writes accepted and next_token.
constexpr int kRowThreadsMax = 1024;
constexpr int kRowLoads = 8;    // vector loads in flight per thread
constexpr int kMaxRowCtas = 8;  // CTAs per row: a portable cluster
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

// VEC = 4: float4 loads (vocab % 4 == 0 and 16-byte aligned logits), else 1.
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
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // a CTA's shared memory may be written by another only once that CTA has
    // started: every CTA arrives here and waits before its remote store
    if (k > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // the logits may come from the kernel before this one
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const int lo = min(rank * a.slice, a.vocab), hi = min(lo + a.slice, a.vocab);
    const int nvec = (hi - lo) / VEC;  // slice is a multiple of VEC
    const float *__restrict__ src = a.logits + row * (size_t)a.vocab + lo;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    const int nt = blockDim.x;
    // batches of kRowLoads vector loads, all issued before the compares
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

// The argmax step: k CTAs per row, k = SMs / rows clamped to [1, 8], with
// enough threads for kRowLoads vector loads each over a 1/k slice.
template <int VEC, bool READOUT>
cudaError_t row_argmax_launch(RowArgs a, long long rows, cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const int sms = attn_grid_size(dev);
    if (sms <= 0) return cudaErrorInvalidDevice;
    const int k = rows >= sms ? 1 : (int)std::min<long long>(kMaxRowCtas, sms / rows);
    const int slice = (a.vocab + k - 1) / k;
    a.slice = (slice + VEC - 1) / VEC * VEC;
    const int nvec = a.slice / VEC;
    int threads = (nvec + kRowLoads - 1) / kRowLoads;
    threads = std::max(32, std::min(kRowThreadsMax, (threads + 31) / 32 * 32));
    if (rows * k > 0x7fffffffLL) return cudaErrorInvalidValue;
    return launch_pdl(row_argmax_kernel<VEC, READOUT>, dim3((unsigned)(rows * k)),
                      dim3((unsigned)threads), (unsigned)k, stream, a);
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

}  // namespace

cudaError_t accept_launch(const float *logits, const int32_t *draft, int B, int W, int vocab,
                          int32_t *accepted, int32_t *target_ids, int32_t *next_token,
                          cudaStream_t stream) {
    RowArgs a = {};
    a.logits = logits;
    a.W = W;
    a.vocab = vocab;
    a.target_ids = target_ids;
    cudaError_t e = argmax_launch(a, B, false, stream);
    if (e != cudaSuccess || B == 0) return e;
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
