// synth_dev.cu -- device side of the seeded input generator (see synth_core.h).
// Built with --fmad=false so that its values equal the host side's bit for
// bit.  Used to fill large caches in place; no method arithmetic lives here.
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth_core.h"

namespace {

// dst: the slab of stored depth `depth`, [layers][batch][capacity][heads][D]
__global__ void fill_matured_kernel(uint16_t *dst, uint64_t key, int is_value, int depth, int R,
                                    int batch, int capacity, int heads, int D, size_t n) {
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        size_t r = idx;
        const uint32_t e = (uint32_t)(r % D);
        r /= D;
        const uint32_t h = (uint32_t)(r % heads);
        r /= heads;
        const uint32_t t = (uint32_t)(r % capacity);
        r /= capacity;
        const uint32_t b = (uint32_t)(r % batch);
        const uint32_t l = (uint32_t)(r / batch);
        dst[idx] = synth_bf16(synth_matured(key, is_value, depth, R, l, b, t, h, e));
    }
}

// Depths the benchmark never reads: cheap values in +-[1, 2) from one hash.
__global__ void fill_filler_kernel(uint16_t *dst, uint64_t key, size_t n) {
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        const uint64_t h = synth_out(key, idx + 1);
        dst[idx] = (uint16_t)(0x3F80u | (h & 0x7Fu) | ((h >> 8) & 1u) << 15);
    }
}

int grid_for(size_t n) {
    int sms = 152;
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    size_t want = (n + 255) / 256;
    size_t cap = (size_t)sms * 16;
    return (int)(want < cap ? (want ? want : 1) : cap);
}

}  // namespace

extern "C" {

// Fill a whole depth slab under the maturation law.  Returns a cudaError_t.
int synth_dev_fill_matured(uint16_t *dst, uint64_t seed, int tensor, int is_value, int depth,
                           int R, int layers, int batch, int capacity, int heads, int D,
                           void *stream) {
    if (depth < 1 || depth > R || R > 63 || layers > 64 || batch > 256 || capacity > (1 << 21) ||
        heads > 256 || D > 512)
        return (int)cudaErrorInvalidValue;
    const size_t n = (size_t)layers * batch * capacity * heads * D;
    if (n == 0) return 0;
    fill_matured_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream>>>(
        dst, synth_key(seed, (uint64_t)tensor), is_value, depth, R, batch, capacity, heads, D, n);
    return (int)cudaGetLastError();
}

int synth_dev_fill_filler(uint16_t *dst, size_t n, uint64_t seed, void *stream) {
    if (n == 0) return 0;
    fill_filler_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream>>>(
        dst, synth_key(seed, SYNTH_T_FILL), n);
    return (int)cudaGetLastError();
}

}  // extern "C"
