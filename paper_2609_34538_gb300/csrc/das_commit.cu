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
// One cluster of CTAS CTAs per sequence (CTAS = 16 for up to four sequences,
// which spreads a sequence's logits over more SMs, else 8: with more
// sequences, 16-CTA clusters measured slower than 8-CTA ones).  CTA r of the
// cluster scans slice r of the vocabulary for every row i < W of its sequence
// and stores its best (value, index) per row straight into CTA 0's shared
// memory (distributed shared memory).  The others then arrive at the cluster
// barrier and exit; CTA 0 waits for them, reduces the CTAS candidates of each
// row from its own shared memory and
//   - accept mode (Sec. 3.4): writes target_ids, counts the accepted prefix
//     and writes accepted and next_token;
//   - readout mode (Eq. 6, Sec. 3.3): writes the argmax of row i as the guess
//     of position i + 1, tokens[b][i + 1].
constexpr int kAcceptThreads = 1024;
constexpr int kAcceptWarps = kAcceptThreads / 32;
constexpr int kMaxW = 1024;
constexpr int kBatch = 8;          // vector loads in flight per thread
constexpr int kWideClusterMaxB = 4;  // sequences up to which a cluster has 16 CTAs

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

// dynamic shared memory of an accept CTA: candidate values [CTAS][W] and
// indices [CTAS][W] (filled in CTA 0 by every CTA), row argmaxes [W] (CTA 0)
__host__ __device__ constexpr size_t accept_smem_bytes(int ctas, int W) {
    return (size_t)ctas * W * 8 + (size_t)W * 4;
}

struct ArgmaxArgs {
    const float *logits;  // [B][W][vocab]
    int W, vocab, slice;
    // accept mode
    const int32_t *draft;
    int32_t *accepted, *target_ids, *next_token;
    // readout mode
    int32_t *tokens;  // [B][stride]
    int stride;
};

// VEC = 4: float4 loads (vocab % 4 == 0 and 16-byte aligned logits), else 1.
template <int VEC, bool READOUT, int CTAS>
__global__ void __launch_bounds__(kAcceptThreads) accept_kernel(const ArgmaxArgs a) {
    const float *__restrict__ logits = a.logits;
    const int W = a.W, vocab = a.vocab, slice = a.slice;
    extern __shared__ __align__(16) uint8_t accept_smem[];
    float *cand_v = reinterpret_cast<float *>(accept_smem);
    int *cand_i = reinterpret_cast<int *>(cand_v + CTAS * W);
    int *target = cand_i + CTAS * W;
    __shared__ float warp_v[kAcceptWarps];
    __shared__ int warp_i[kAcceptWarps];
    __shared__ int first_miss;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int b = blockIdx.x / CTAS;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // a CTA's shared memory may be written by another only once that CTA has
    // started: every CTA arrives here and waits before its first remote store
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    float *dst_v = cluster.map_shared_rank(cand_v, 0) + rank * W;
    int *dst_i = cluster.map_shared_rank(cand_i, 0) + rank * W;

    // threads per row: the CTA's warps split over min(W, 32) rows at a time
    int tpr = kAcceptThreads;
    while (tpr > 32 && tpr * W > kAcceptThreads) tpr >>= 1;
    const int rows_per_pass = kAcceptThreads / tpr, warps_per_row = tpr / 32;
    const int lo = min(rank * slice, vocab), hi = min(lo + slice, vocab);
    const int nvec = (hi - lo) / VEC;  // slice is a multiple of VEC
    for (int i0 = 0; i0 < W; i0 += rows_per_pass) {
        const int i = i0 + threadIdx.x / tpr;
        const int part = threadIdx.x % tpr;
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        if (i < W) {
            const float *row = logits + ((size_t)b * W + i) * (size_t)vocab + lo;
            // batches of kBatch vector loads, all issued before the compares
            for (int j0 = part; j0 < nvec; j0 += kBatch * tpr) {
                float x[kBatch][VEC];
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const int j = j0 + u * tpr;
                    if (j < nvec) {
                        if (VEC == 4) {
                            const float4 y = __ldcs(reinterpret_cast<const float4 *>(row) + j);
                            x[u][0] = y.x;
                            x[u][1 % VEC] = y.y;
                            x[u][2 % VEC] = y.z;
                            x[u][VEC - 1] = y.w;
                        } else {
                            x[u][0] = __ldcs(row + j);
                        }
                    }
                }
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const int j = j0 + u * tpr;
                    if (j < nvec) {
#pragma unroll
                        for (int e = 0; e < VEC; ++e) better(bv, bi, x[u][e], lo + VEC * j + e);
                    }
                }
            }
        }
        warp_best(bv, bi);
        if (lane == 0) {
            warp_v[warp] = bv;
            warp_i[warp] = bi;
        }
        __syncthreads();
        if (i0 == 0) asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
        if (threadIdx.x < rows_per_pass && i0 + (int)threadIdx.x < W) {
            float v = -INFINITY;
            int y = 0x7fffffff;
            for (int w = 0; w < warps_per_row; ++w)
                better(v, y, warp_v[threadIdx.x * warps_per_row + w],
                       warp_i[threadIdx.x * warps_per_row + w]);
            dst_v[i0 + threadIdx.x] = v;
            dst_i[i0 + threadIdx.x] = y;
        }
        __syncthreads();
    }
    // the candidates are in CTA 0 once every CTA has arrived (release); only
    // CTA 0 waits, and no CTA's shared memory but CTA 0's is ever read remotely
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    if (rank != 0) return;
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");

    if (threadIdx.x == 0) first_miss = W;
    __syncthreads();
    for (int i = threadIdx.x; i < W; i += kAcceptThreads) {
        float v = -INFINITY;
        int x = 0x7fffffff;
#pragma unroll
        for (int r = 0; r < CTAS; ++r) better(v, x, cand_v[r * W + i], cand_i[r * W + i]);
        // a row of -inf keeps the sentinel: the first index wins
        const int t = x == 0x7fffffff ? 0 : x;
        if (READOUT) {
            a.tokens[(size_t)b * a.stride + i + 1] = t;
        } else {
            target[i] = t;
            a.target_ids[(size_t)b * W + i] = t;
            if (a.draft[(size_t)b * W + i] != t) atomicMin(&first_miss, i);
        }
    }
    if (!READOUT) {
        __syncthreads();
        if (threadIdx.x == 0) {
            const int n = first_miss;
            a.accepted[b] = n;
            a.next_token[b] = n < W ? target[n] : a.draft[(size_t)b * W + W - 1];
        }
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

// The dynamic shared memory opt-in (and, for 16-CTA clusters, the non-portable
// cluster size) of one accept kernel, once per device.  Returns false if the
// kernel cannot run with that many CTAs per cluster on this device.
template <int VEC, bool READOUT, int CTAS>
cudaError_t accept_configure(int dev, bool &usable) {
    static std::atomic<int> state[64];  // 0 unknown, 1 usable, 2 not usable
    usable = false;
    if (dev < 64) {
        const int st = state[dev].load(std::memory_order_acquire);
        if (st != 0) {
            usable = st == 1;
            return cudaSuccess;
        }
    }
    auto kernel = accept_kernel<VEC, READOUT, CTAS>;
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)accept_smem_bytes(CTAS, kMaxW));
    if (e != cudaSuccess) return e;
    if (CTAS > 8) {
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(CTAS);
        cfg.blockDim = dim3(kAcceptThreads);
        cfg.dynamicSmemBytes = accept_smem_bytes(CTAS, kMaxW);
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = CTAS;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        int clusters = 0;
        e = cudaOccupancyMaxActiveClusters(&clusters, kernel, &cfg);
        if (e != cudaSuccess) return e;
        usable = clusters >= 1;
    } else {
        usable = true;
    }
    if (dev < 64) state[dev].store(usable ? 1 : 2, std::memory_order_release);
    return cudaSuccess;
}

template <int VEC, bool READOUT, int CTAS>
cudaError_t argmax_launch_ctas(ArgmaxArgs a, int B, cudaStream_t stream) {
    // slices are whole float4s
    const int slice = (a.vocab + CTAS - 1) / CTAS;
    a.slice = (slice + 3) & ~3;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(B * CTAS));
    cfg.blockDim = dim3(kAcceptThreads);
    cfg.dynamicSmemBytes = accept_smem_bytes(CTAS, a.W);
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = CTAS;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, accept_kernel<VEC, READOUT, CTAS>, a);
}

template <int VEC, bool READOUT>
cudaError_t argmax_launch_vec(const ArgmaxArgs &a, int B, cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    bool usable = false;
    if (B <= kWideClusterMaxB) {
        e = accept_configure<VEC, READOUT, 16>(dev, usable);
        if (e != cudaSuccess) return e;
        if (usable) return argmax_launch_ctas<VEC, READOUT, 16>(a, B, stream);
    }
    e = accept_configure<VEC, READOUT, 8>(dev, usable);
    if (e != cudaSuccess) return e;
    return argmax_launch_ctas<VEC, READOUT, 8>(a, B, stream);
}

cudaError_t argmax_launch(const ArgmaxArgs &a, int B, bool readout, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if (a.W < 1 || a.W > kMaxW || B > 0x7fffffff / 16) return cudaErrorInvalidValue;
    const bool vec = (a.vocab % 4) == 0 && (reinterpret_cast<uintptr_t>(a.logits) & 15u) == 0;
    if (readout)
        return vec ? argmax_launch_vec<4, true>(a, B, stream)
                   : argmax_launch_vec<1, true>(a, B, stream);
    return vec ? argmax_launch_vec<4, false>(a, B, stream)
               : argmax_launch_vec<1, false>(a, B, stream);
}

}  // namespace

cudaError_t accept_launch(const float *logits, const int32_t *draft, int B, int W, int vocab,
                          int32_t *accepted, int32_t *target_ids, int32_t *next_token,
                          cudaStream_t stream) {
    ArgmaxArgs a = {};
    a.logits = logits;
    a.W = W;
    a.vocab = vocab;
    a.draft = draft;
    a.accepted = accepted;
    a.target_ids = target_ids;
    a.next_token = next_token;
    return argmax_launch(a, B, false, stream);
}

cudaError_t wave_readout_launch(const float *logits, int B, int W, int vocab, int32_t *tokens,
                                int stride, cudaStream_t stream) {
    ArgmaxArgs a = {};
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
