// das_internal.h -- declarations shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "das.h"

namespace das {

// Work unit of the attention kernels: 64 key positions of one (sequence, kv
// head).  Every (sequence, kv head) pair owns ceil(P/64) prefix tiles plus one
// tile for the draft block's own keys.
constexpr int kTileKeys = 64;
constexpr int kMaxRows = 64;          // G * max_block handled by one pair
constexpr size_t kWorkspaceHeader = 256;

// Bits of the workspace status word.
constexpr int kStatusWaitTimeout = 1;
constexpr int kStatusClamped = 2;

struct AttnParams {
    const int32_t *prefix_len;
    const int32_t *block_len;
    const uint16_t *q;  // bf16 [B][max_block][Hq][D]
    uint16_t *out;      // bf16 [B][max_block][Hq][D]
    float *lse;         // [B][Hq][max_block]
    float *part_o;      // [slots][rows_max][D]
    float *part_lse;    // [slots][rows_max]
    int32_t *status;    // workspace status word
    int B, Hq, Hkv, G, max_block, rows_max, capacity;
    int key_slab, value_slab;  // (depth - 1) * layers + layer
    float scale_log2;          // softmax scale * log2(e)
    int num_ctas;
};

// Number of CTAs the attention kernel launches on `device` (a persistent
// grid, one CTA per SM).
int attn_grid_size(int device);
size_t attn_workspace_bytes(int device, int batch, int kv_heads, int rows_max, int head_dim);
// Carve a workspace into status word and partials (sets p.status, p.part_o,
// p.part_lse).
void attn_workspace_layout(void *workspace, int batch, int kv_heads, int rows_max, int head_dim,
                           int num_ctas, AttnParams &p);

// Launch the tcgen05 attention kernel and its split-K merge on `stream`, each
// a programmatic dependent of the kernel before it; tm_q maps the queries
// [B][max_block][Hq][D] with a {64, G, max_block, 1} box.
// keys_e4m3 / values_e4m3: tm_k / tm_v map e4m3 prefix tiles (8-bit maps with
// a {D, 1, 64, 1, 1} box, no swizzle) instead of bf16 ones.
cudaError_t attn_launch(const AttnParams &p, int head_dim, bool keys_e4m3, bool values_e4m3,
                        const CUtensorMap &tm_k, const CUtensorMap &tm_v,
                        const CUtensorMap &tm_kb, const CUtensorMap &tm_vb,
                        const CUtensorMap &tm_q, cudaStream_t stream);

// das_mature_v_attention (key_depth = value_depth for the verify attention)
// with every argument checked; with clear_status, the workspace's 256-byte
// header is zeroed on `stream` after the checks pass, right before the
// launch (nothing is enqueued for a call that returns an error).
das_status attention(const das_kv_cache *c, int layer, int key_depth, int value_depth,
                     const int32_t *prefix_len, const int32_t *block_len, int max_block,
                     const void *q, const void *k_blk, const void *v_blk, int num_q_heads,
                     float softmax_scale, void *out, float *lse, void *workspace,
                     size_t workspace_bytes, bool clear_status, void *stream);

cudaError_t accept_launch(const float *logits, const int32_t *draft, int B, int W, int vocab,
                          int32_t *accepted, int32_t *target_ids, int32_t *next_token,
                          cudaStream_t stream);

// tokens[b][i + 1] = argmax of logits[b][i] for i < W (Eq. 6 readout).
cudaError_t wave_readout_launch(const float *logits, int B, int W, int vocab, int32_t *tokens,
                                int stride, cudaStream_t stream);

cudaError_t append_launch(const das_kv_cache &c, const void *k_new, const void *v_new,
                          const int32_t *accepted, int W, int32_t *prefix_len,
                          int32_t *error_flag, cudaStream_t stream);

// das_kv_append_f8: depth R copied to the bf16 top tensors, depths below R
// rounded to e4m3 into the low tensors.
cudaError_t append_f8_launch(const das_kv_cache_f8 &c, const void *k_new, const void *v_new,
                             const int32_t *accepted, int W, int32_t *prefix_len,
                             int32_t *error_flag, cudaStream_t stream);

}  // namespace das
