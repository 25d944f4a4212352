// das_commit.cu -- greedy acceptance and the multi-depth cache commit
// (Sec. 3.4; App. B.1) on sm_103a.
#include "das_internal.h"

namespace das {
namespace {

constexpr int kArgmaxThreads = 512;

// (value, index) order of the argmax: larger value wins, equal values go to
// the smaller index, so the result is the first maximum.
__device__ __forceinline__ void better(float &bv, int &bi, float v, int i) {
    if (v > bv || (v == bv && i < bi)) {
        bv = v;
        bi = i;
    }
}

// One CTA per (sequence, proposal) row: target_ids[b][i] = argmax over vocab.
__global__ void __launch_bounds__(kArgmaxThreads) argmax_kernel(const float *__restrict__ logits,
                                                                int vocab,
                                                                int32_t *__restrict__ target_ids) {
    const size_t row = blockIdx.x;
    const float *x = logits + row * (size_t)vocab;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    const bool vec = (vocab & 3) == 0;
    if (vec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(x);
        const int n4 = vocab >> 2;
        int j = threadIdx.x;
        for (; j + 3 * kArgmaxThreads < n4; j += 4 * kArgmaxThreads) {
            float4 a[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) a[u] = __ldcs(x4 + j + u * kArgmaxThreads);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int base = 4 * (j + u * kArgmaxThreads);
                better(bv, bi, a[u].x, base);
                better(bv, bi, a[u].y, base + 1);
                better(bv, bi, a[u].z, base + 2);
                better(bv, bi, a[u].w, base + 3);
            }
        }
        for (; j < n4; j += kArgmaxThreads) {
            const float4 a = __ldcs(x4 + j);
            better(bv, bi, a.x, 4 * j);
            better(bv, bi, a.y, 4 * j + 1);
            better(bv, bi, a.z, 4 * j + 2);
            better(bv, bi, a.w, 4 * j + 3);
        }
    } else {
        for (int j = threadIdx.x; j < vocab; j += kArgmaxThreads) better(bv, bi, __ldcs(x + j), j);
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, d);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, d);
        better(bv, bi, ov, oi);
    }
    __shared__ float sv[kArgmaxThreads / 32];
    __shared__ int si[kArgmaxThreads / 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        sv[warp] = bv;
        si[warp] = bi;
    }
    __syncthreads();
    if (warp == 0) {
        bv = lane < kArgmaxThreads / 32 ? sv[lane] : -INFINITY;
        bi = lane < kArgmaxThreads / 32 ? si[lane] : 0x7fffffff;
#pragma unroll
        for (int d = 16; d > 0; d >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, d);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, d);
            better(bv, bi, ov, oi);
        }
        // A row of -inf only keeps bi at its sentinel: the first index wins.
        if (lane == 0) target_ids[row] = bi == 0x7fffffff ? 0 : bi;
    }
}

// accepted[b] = leading matches; next_token[b] as in Sec. 3.4.
__global__ void accept_count_kernel(const int32_t *__restrict__ draft,
                                    const int32_t *__restrict__ target_ids, int B, int W,
                                    int32_t *__restrict__ accepted, int32_t *__restrict__ next) {
    for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < B; b += gridDim.x * blockDim.x) {
        const int32_t *d = draft + (size_t)b * W;
        const int32_t *t = target_ids + (size_t)b * W;
        int a = 0;
        while (a < W && d[a] == t[a]) ++a;
        accepted[b] = a;
        next[b] = a < W ? t[a] : d[W - 1];
    }
}

__device__ __forceinline__ int append_count(int32_t a, int W) {
    if (a < 0) a = 0;
    return a + 1 < W ? a + 1 : W;
}

// Copy the materialized inputs' K/V of slab (depth, layer, b): blockIdx.x is
// (depth * layers + layer) * batch + b.  Each 16-byte word is one vector copy.
__global__ void append_copy_kernel(uint4 *__restrict__ kc, uint4 *__restrict__ vc,
                                   const uint4 *__restrict__ kn, const uint4 *__restrict__ vn,
                                   const int32_t *__restrict__ accepted,
                                   const int32_t *__restrict__ prefix_len, int batch, int capacity,
                                   int W, int row_words) {
    const int slab = blockIdx.x;
    const int b = slab % batch;
    const int n = append_count(accepted[b], W);
    const int p = prefix_len[b];
    if (p < 0 || p + n > capacity) return;  // reported by append_finalize_kernel
    const size_t words = (size_t)n * row_words;
    const uint4 *ks = kn + (size_t)slab * W * row_words;
    const uint4 *vs = vn + (size_t)slab * W * row_words;
    uint4 *kd = kc + ((size_t)slab * capacity + p) * row_words;
    uint4 *vd = vc + ((size_t)slab * capacity + p) * row_words;
    for (size_t i = threadIdx.x; i < words; i += blockDim.x) {
        kd[i] = __ldcs(ks + i);
        vd[i] = __ldcs(vs + i);
    }
}

// Runs after every copy: grow prefix_len or flag the sequence.
__global__ void append_finalize_kernel(const int32_t *__restrict__ accepted,
                                       int32_t *__restrict__ prefix_len, int batch, int capacity,
                                       int W, int32_t *__restrict__ error_flag) {
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

}  // namespace

cudaError_t accept_launch(const float *logits, const int32_t *draft, int B, int W, int vocab,
                          int32_t *accepted, int32_t *target_ids, int32_t *next_token,
                          cudaStream_t stream) {
    if (B == 0) return cudaSuccess;
    argmax_kernel<<<B * W, kArgmaxThreads, 0, stream>>>(logits, vocab, target_ids);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    accept_count_kernel<<<(B + 127) / 128, 128, 0, stream>>>(draft, target_ids, B, W, accepted,
                                                            next_token);
    return cudaGetLastError();
}

cudaError_t append_launch(const das_kv_cache &c, const void *k_new, const void *v_new,
                          const int32_t *accepted, int W, int32_t *prefix_len,
                          int32_t *error_flag, cudaStream_t stream) {
    const int row_words = c.kv_heads * c.head_dim * 2 / 16;
    const int slabs = c.depths * c.layers * c.batch;
    if (slabs == 0) return cudaSuccess;
    append_copy_kernel<<<slabs, 256, 0, stream>>>(
        static_cast<uint4 *>(c.k), static_cast<uint4 *>(c.v), static_cast<const uint4 *>(k_new),
        static_cast<const uint4 *>(v_new), accepted, prefix_len, c.batch, c.capacity, W,
        row_words);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    append_finalize_kernel<<<(c.batch + 127) / 128, 128, 0, stream>>>(accepted, prefix_len,
                                                                      c.batch, c.capacity, W,
                                                                      error_flag);
    return cudaGetLastError();
}

}  // namespace das
