// das_noalloc.cu -- a variant of das_mature_v_attention that needs no
// workspace from its caller.
//
// Some callers cannot allocate device memory at the point where they call
// the library: code that runs under an allocator that must not grow (a
// serving loop with a fixed memory plan), plugins that are handed only the
// tensors they operate on, or hosts that forbid cudaMalloc after start-up.
// For them, this entry point keeps its split-K scratch in a fixed array that
// is part of the library's device image: it is created when the library's
// module is loaded on a device and stays there until the process exits.
//
// The scratch is shared by every call on a device, so calls that overlap in
// time on the GPU (on different streams) race on it; callers must order
// them.  Its contents persist between calls; the only part that must start at
// zero (the status word at its head) is cleared by every call that passes
// its argument checks, just before its kernels are launched.
//
// The array's device address is looked up once per device (a host-side name
// of a __device__ variable is not a device address) and kept for the
// process; a call after the device's primary context was destroyed
// (cudaDeviceReset) would use a stale address, so such a reset ends the use
// of this entry point in that process.
#include <mutex>

#include "das_internal.h"

namespace {

// Largest split-K workspace this entry point can serve.
constexpr size_t kScratchBytes = DAS_NOALLOC_SCRATCH_BYTES;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_mu;
void *g_scratch_ptr[64] = {nullptr};  // device address of g_scratch per device

// Device address of g_scratch on the current device (set-up on first use).
void *scratch_address(int dev) {
    if (dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess) return nullptr;
        g_scratch_ptr[dev] = ptr;
    }
    return g_scratch_ptr[dev];
}

}  // namespace

extern "C" das_status das_mature_v_attention_noalloc(
    const das_kv_cache *cache, int layer, int key_depth, int value_depth,
    const int32_t *prefix_len, const int32_t *block_len, int max_block, const void *q,
    const void *k_blk, const void *v_blk, int num_q_heads, float softmax_scale, void *out,
    float *lse, void *stream) {
    const size_t need = das_workspace_size(cache, num_q_heads, max_block);
    if (need > kScratchBytes) return DAS_ERR_WORKSPACE;
    if (need == 0)  // unsupported or invalid shape: let the full check report it
        return das::attention(cache, layer, key_depth, value_depth, prefix_len, block_len,
                              max_block, q, k_blk, v_blk, num_q_heads, softmax_scale, out, lse,
                              nullptr, 0, false, stream);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DAS_ERR_CUDA;
    void *ws = scratch_address(dev);
    if (!ws) return DAS_ERR_CUDA;
    // the status word must start at zero for this call: the attention path
    // clears it once every argument has been checked, just before its launch
    return das::attention(cache, layer, key_depth, value_depth, prefix_len, block_len, max_block,
                          q, k_blk, v_blk, num_q_heads, softmax_scale, out, lse, ws, kScratchBytes,
                          true, stream);
}

extern "C" das_status das_noalloc_status(int32_t *dst, void *stream) {
    if (!dst) return DAS_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DAS_ERR_CUDA;
    void *ws = scratch_address(dev);
    if (!ws) return DAS_ERR_CUDA;
    return cudaMemcpyAsync(dst, ws, sizeof(int32_t), cudaMemcpyDefault,
                           static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAS_OK
               : DAS_ERR_CUDA;
}
