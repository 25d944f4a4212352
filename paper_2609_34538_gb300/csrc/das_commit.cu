// das_commit.cu -- greedy acceptance and the multi-depth cache commit
// (Sec. 3.4; App. B.1) on sm_103a.
//
// Every kernel here is launched as a programmatic dependent of the previous
// kernel in the stream: it reads nothing before griddepcontrol.wait, and
// every CTA executes that wait.
#include <cooperative_groups.h>

#include "das_internal.h"

namespace cg = cooperative_groups;

namespace das {
namespace {

// ---- greedy acceptance and the DAS-Wave readout ------------------------------
// One cluster of kAcceptCtas CTAs per sequence.  CTA j of the cluster scans
// slice j of the vocabulary for every row i < W of its sequence and keeps its
// best (value, index) per row in shared memory; after a cluster barrier CTA 0
// reads the kAcceptCtas candidates of each row through distributed shared
// memory and
//   - accept mode (Sec. 3.4): writes target_ids, counts the accepted prefix
//     and writes accepted and next_token;
//   - readout mode (Eq. 6, Sec. 3.3): writes the argmax of row i as the guess
//     of position i + 1, tokens[b][i + 1].
constexpr int kAcceptCtas = 8;
constexpr int kAcceptThreads = 1024;
constexpr int kAcceptWarps = kAcceptThreads / 32;
constexpr int kMaxW = 1024;
constexpr int kBatch = 8;  // vector loads in flight per thread

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

struct AcceptSmem {
    float cand_v[kMaxW];  // this CTA's best per row
    int cand_i[kMaxW];
    float warp_v[kAcceptWarps];
    int warp_i[kAcceptWarps];
    int target[kMaxW];  // CTA 0: the row argmaxes
    int first_miss;
};

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
template <int VEC, bool READOUT>
__global__ void __launch_bounds__(kAcceptThreads) accept_kernel(const ArgmaxArgs a) {
    const float *__restrict__ logits = a.logits;
    const int W = a.W, vocab = a.vocab, slice = a.slice;
    __shared__ AcceptSmem sm;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int b = blockIdx.x / kAcceptCtas;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

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
                float a[kBatch][VEC];
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const int j = j0 + u * tpr;
                    if (j < nvec) {
                        if (VEC == 4) {
                            const float4 x = __ldcs(reinterpret_cast<const float4 *>(row) + j);
                            a[u][0] = x.x;
                            a[u][1 % VEC] = x.y;
                            a[u][2 % VEC] = x.z;
                            a[u][VEC - 1] = x.w;
                        } else {
                            a[u][0] = __ldcs(row + j);
                        }
                    }
                }
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    const int j = j0 + u * tpr;
                    if (j < nvec) {
#pragma unroll
                        for (int e = 0; e < VEC; ++e) better(bv, bi, a[u][e], lo + VEC * j + e);
                    }
                }
            }
        }
        warp_best(bv, bi);
        if (lane == 0) {
            sm.warp_v[warp] = bv;
            sm.warp_i[warp] = bi;
        }
        __syncthreads();
        if (threadIdx.x < rows_per_pass && i0 + (int)threadIdx.x < W) {
            float v = -INFINITY;
            int x = 0x7fffffff;
            for (int w = 0; w < warps_per_row; ++w)
                better(v, x, sm.warp_v[threadIdx.x * warps_per_row + w],
                       sm.warp_i[threadIdx.x * warps_per_row + w]);
            sm.cand_v[i0 + threadIdx.x] = v;
            sm.cand_i[i0 + threadIdx.x] = x;
        }
        __syncthreads();
    }
    cluster.sync();  // every CTA's candidates are in its shared memory

    if (rank == 0) {
        if (threadIdx.x == 0) sm.first_miss = W;
        __syncthreads();
        for (int i = threadIdx.x; i < W; i += kAcceptThreads) {
            float v = -INFINITY;
            int x = 0x7fffffff;
#pragma unroll
            for (int r = 0; r < kAcceptCtas; ++r) {
                const AcceptSmem *o = cluster.map_shared_rank(&sm, r);
                better(v, x, o->cand_v[i], o->cand_i[i]);
            }
            // a row of -inf keeps the sentinel: the first index wins
            const int t = x == 0x7fffffff ? 0 : x;
            if (READOUT) {
                a.tokens[(size_t)b * a.stride + i + 1] = t;
            } else {
                sm.target[i] = t;
                a.target_ids[(size_t)b * W + i] = t;
                if (a.draft[(size_t)b * W + i] != t) atomicMin(&sm.first_miss, i);
            }
        }
        if (!READOUT) {
            __syncthreads();
            if (threadIdx.x == 0) {
                const int n = sm.first_miss;
                a.accepted[b] = n;
                a.next_token[b] = n < W ? sm.target[n] : a.draft[(size_t)b * W + W - 1];
            }
        }
    }
    cluster.sync();  // CTA 0 has read the others' shared memory
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

cudaError_t argmax_launch(const ArgmaxArgs &a0, int B, bool readout, cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    if (a0.W > kMaxW || B > 0x7fffffff / kAcceptCtas) return cudaErrorInvalidValue;
    ArgmaxArgs a = a0;
    const bool vec = (a.vocab % 4) == 0 && (reinterpret_cast<uintptr_t>(a.logits) & 15u) == 0;
    // slices are whole float4s
    int slice = (a.vocab + kAcceptCtas - 1) / kAcceptCtas;
    a.slice = (slice + 3) & ~3;
    const dim3 grid((unsigned)(B * kAcceptCtas)), block(kAcceptThreads);
    if (readout)
        return vec ? launch_pdl(accept_kernel<4, true>, grid, block, kAcceptCtas, stream, a)
                   : launch_pdl(accept_kernel<1, true>, grid, block, kAcceptCtas, stream, a);
    return vec ? launch_pdl(accept_kernel<4, false>, grid, block, kAcceptCtas, stream, a)
               : launch_pdl(accept_kernel<1, false>, grid, block, kAcceptCtas, stream, a);
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
