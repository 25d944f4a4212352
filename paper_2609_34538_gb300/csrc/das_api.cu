// das_api.cu -- the library's C ABI (include/das.h): argument checks, TMA
// tensor-map encoding and launches.  Nothing here allocates device memory.
#include <math.h>
#include <mutex>

#include "das_internal.h"

namespace das {
namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Tensor map over `rank` dims (innermost first): bf16 elements with 128-byte
// swizzle, or 8-bit (e4m3) elements without swizzle (their tiles are widened
// by the kernel, which reads them row by row) or, with swizzle8, with 128-byte
// swizzle (key tiles of 128-byte rows that the e4m3 MMAs read as they land).
bool encode_uncached(CUtensorMap *m, void *base, int rank, const cuuint64_t *dims,
                     const cuuint32_t *box, bool e4m3, bool swizzle8) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t strides[4];
    cuuint64_t s = e4m3 ? 1 : 2;
    for (int i = 0; i < rank - 1; ++i) {
        s *= dims[i];
        strides[i] = s;
    }
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    // L2 promotion no wider than one contiguous row: the rows of one head are
    // strided by the other heads, so a 256-byte promotion of a 128-byte row
    // (an e4m3 row of 128 dims, a bf16 row of 64) fetches a neighbour's row too.
    const cuuint64_t row_bytes = dims[0] * (e4m3 ? 1 : 2);
    const CUtensorMapL2promotion promo = row_bytes >= 256   ? CU_TENSOR_MAP_L2_PROMOTION_L2_256B
                                         : row_bytes >= 128 ? CU_TENSOR_MAP_L2_PROMOTION_L2_128B
                                                            : CU_TENSOR_MAP_L2_PROMOTION_L2_64B;
    return fn(m, e4m3 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
              (cuuint32_t)rank, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              e4m3 && !swizzle8 ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_128B, promo,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded maps are kept in a small direct-mapped table keyed by everything
// the encoding depends on (address, rank, extents, box): a serving loop calls
// with the same buffers every step, and an encode costs about as much host
// time as a launch.  A hit returns a copy of the very descriptor an encode
// would produce, so the table never changes a result.
struct MapKey {
    void *base;
    int rank;
    bool e4m3, swizzle8;
    cuuint64_t dims[5];
    cuuint32_t box[5];
};
struct MapSlot {
    bool used;
    MapKey key;
    CUtensorMap map;
};
constexpr int kMapSlots = 256;
std::mutex g_map_mu;
MapSlot g_maps[kMapSlots];

bool same_key(const MapKey &a, const MapKey &b) {
    if (a.base != b.base || a.rank != b.rank || a.e4m3 != b.e4m3 || a.swizzle8 != b.swizzle8)
        return false;
    for (int i = 0; i < a.rank; ++i)
        if (a.dims[i] != b.dims[i] || a.box[i] != b.box[i]) return false;
    return true;
}

bool encode(CUtensorMap *m, void *base, int rank, const cuuint64_t *dims,
            const cuuint32_t *box_in, bool e4m3, bool swizzle8 = false) {
    MapKey key = {};
    key.base = base;
    key.rank = rank;
    key.e4m3 = e4m3;
    key.swizzle8 = swizzle8;
    const cuuint32_t box_default[5] = {64, 1, 64, 1, 1};
    for (int i = 0; i < rank; ++i) {
        key.dims[i] = dims[i];
        key.box[i] = box_in ? box_in[i] : box_default[i];
    }
    uint64_t h = 1469598103934665603ull;  // FNV-1a over the key's fields
    auto mix = [&h](uint64_t v) {
        for (int i = 0; i < 8; ++i) {
            h ^= (v >> (8 * i)) & 0xffu;
            h *= 1099511628211ull;
        }
    };
    mix(reinterpret_cast<uintptr_t>(base));
    mix((uint64_t)rank * 4 + (e4m3 ? 1 : 0) + (swizzle8 ? 2 : 0));
    for (int i = 0; i < rank; ++i) {
        mix(key.dims[i]);
        mix(key.box[i]);
    }
    MapSlot &slot = g_maps[h % kMapSlots];
    {
        std::lock_guard<std::mutex> lock(g_map_mu);
        if (slot.used && same_key(slot.key, key)) {
            *m = slot.map;
            return true;
        }
    }
    if (!encode_uncached(m, base, rank, key.dims, key.box, e4m3, swizzle8)) return false;
    std::lock_guard<std::mutex> lock(g_map_mu);
    slot.used = true;
    slot.key = key;
    slot.map = *m;
    return true;
}

bool encode_bf16(CUtensorMap *m, void *base, int rank, const cuuint64_t *dims,
                 const cuuint32_t *box_in = nullptr) {
    return encode(m, base, rank, dims, box_in, false);
}

bool cache_ok(const das_kv_cache *c) {
    return c && c->k && c->v && c->depths >= 1 && c->depths <= 63 && c->layers >= 1 &&
           c->batch >= 1 && c->capacity >= 1 && c->kv_heads >= 1 &&
           (c->head_dim == 64 || c->head_dim == 128) && aligned16(c->k) && aligned16(c->v);
}

bool cache_f8_ok(const das_kv_cache_f8 *c) {
    return c && c->k_top && c->v_top && c->depths >= 1 && c->depths <= 63 && c->layers >= 1 &&
           c->batch >= 1 && c->capacity >= 1 && c->kv_heads >= 1 &&
           (c->head_dim == 64 || c->head_dim == 128) && aligned16(c->k_top) &&
           aligned16(c->v_top) &&
           (c->depths == 1 || (c->k_low && c->v_low && aligned16(c->k_low) && aligned16(c->v_low)));
}

// The prefix K or V one call reads: a tensor [slabs][batch][capacity][Hkv][D]
// of bf16 or e4m3 elements, and the slab ((depth - 1) * layers + layer).
struct Operand {
    void *base;
    bool e4m3;
    int slabs, slab;
};

// Shape shared by both cache kinds.
struct Shape {
    int depths, layers, batch, capacity, kv_heads, head_dim;
};

das_status attention_core(const Shape &c, int layer, Operand key, Operand value,
                          const int32_t *prefix_len, const int32_t *block_len, int max_block,
                          const void *q, const void *k_blk, const void *v_blk, int num_q_heads,
                          float softmax_scale, void *out, float *lse, void *workspace,
                          size_t workspace_bytes, bool clear_status, void *stream) {
    if (layer < 0 || layer >= c.layers || !prefix_len || !block_len || !q || !k_blk || !v_blk ||
        !out || !lse || num_q_heads < 1 || max_block < 1 || num_q_heads % c.kv_heads != 0 ||
        !aligned16(q) || !aligned16(k_blk) || !aligned16(v_blk) || !aligned16(out) ||
        !isfinite(softmax_scale))
        return DAS_ERR_INVALID_ARG;
    const int G = num_q_heads / c.kv_heads;
    if (max_block > kTileKeys || (long long)G * max_block > kMaxRows) return DAS_ERR_UNSUPPORTED;
    if ((long long)c.capacity > (1ll << 31) / 2 || c.batch > (1 << 20))
        return DAS_ERR_UNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return DAS_ERR_CUDA;
    const size_t need = attn_workspace_bytes(dev, c.batch, c.kv_heads, G * max_block, c.head_dim);
    if (need == 0) return DAS_ERR_CUDA;
    if (!workspace || workspace_bytes < need ||
        (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return DAS_ERR_WORKSPACE;

    const int D = c.head_dim;
    CUtensorMap tk, tv, tkb, tvb, tq;
    auto operand_map = [&](CUtensorMap *m, const Operand &o, bool swizzle8) {
        const cuuint64_t dims[5] = {(cuuint64_t)D, (cuuint64_t)c.kv_heads, (cuuint64_t)c.capacity,
                                    (cuuint64_t)c.batch, (cuuint64_t)o.slabs};
        // e4m3: one {D, 1, 64} box per tile; bf16: {64, 1, 64} swizzled panels
        const cuuint32_t box8[5] = {(cuuint32_t)D, 1, 64, 1, 1};
        return encode(m, o.base, 5, dims, o.e4m3 ? box8 : nullptr, o.e4m3, swizzle8);
    };
    // e4m3 keys with bf16 values at D = 128 are read by the e4m3 MMAs straight
    // from the 128-byte-swizzled tile (the kernel's query-split path)
    const bool key_swizzle8 = key.e4m3 && !value.e4m3 && D == 128;
    const cuuint64_t blk_dims[4] = {(cuuint64_t)D, (cuuint64_t)c.kv_heads, (cuuint64_t)max_block,
                                    (cuuint64_t)c.batch};
    if (!operand_map(&tk, key, key_swizzle8) || !operand_map(&tv, value, false) ||
        !encode_bf16(&tkb, const_cast<void *>(k_blk), 4, blk_dims) ||
        !encode_bf16(&tvb, const_cast<void *>(v_blk), 4, blk_dims))
        return DAS_ERR_CUDA;
    // queries: rows of one pair are heads h*G .. h*G+G-1 of every block row i,
    // i.e. a {64, G, max_block, 1} box over [B][max_block][Hq][D]
    const cuuint64_t q_dims[4] = {(cuuint64_t)D, (cuuint64_t)num_q_heads, (cuuint64_t)max_block,
                                  (cuuint64_t)c.batch};
    const cuuint32_t q_box[4] = {64, (cuuint32_t)G, (cuuint32_t)max_block, 1};
    if (!encode_bf16(&tq, const_cast<void *>(q), 4, q_dims, q_box)) return DAS_ERR_CUDA;

    AttnParams p;
    p.prefix_len = prefix_len;
    p.block_len = block_len;
    p.q = static_cast<const uint16_t *>(q);
    p.out = static_cast<uint16_t *>(out);
    p.lse = lse;
    p.B = c.batch;
    p.Hq = num_q_heads;
    p.Hkv = c.kv_heads;
    p.G = G;
    p.max_block = max_block;
    p.rows_max = G * max_block;
    p.capacity = c.capacity;
    p.key_slab = key.slab;
    p.value_slab = value.slab;
    const double scale = softmax_scale > 0.f ? (double)softmax_scale : 1.0 / sqrt((double)D);
    p.scale_log2 = (float)(scale * 1.4426950408889634);
    p.num_ctas = attn_grid_size(dev);
    attn_workspace_layout(workspace, c.batch, c.kv_heads, p.rows_max, D, p.num_ctas, p);
    // every argument is valid from here on: the only work before the launch
    if (clear_status && cudaMemsetAsync(workspace, 0, kWorkspaceHeader,
                                        static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return DAS_ERR_CUDA;
    const cudaError_t e = attn_launch(p, D, key.e4m3, value.e4m3, tk, tv, tkb, tvb, tq,
                                      static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? DAS_OK : DAS_ERR_CUDA;
}

}  // namespace

das_status attention(const das_kv_cache *c, int layer, int key_depth, int value_depth,
                     const int32_t *prefix_len, const int32_t *block_len, int max_block,
                     const void *q, const void *k_blk, const void *v_blk, int num_q_heads,
                     float softmax_scale, void *out, float *lse, void *workspace,
                     size_t workspace_bytes, bool clear_status, void *stream) {
    if (!cache_ok(c)) {
        if (c && c->head_dim != 64 && c->head_dim != 128 && c->k && c->v) return DAS_ERR_UNSUPPORTED;
        return DAS_ERR_INVALID_ARG;
    }
    if (key_depth < 1 || key_depth > c->depths || value_depth < 1 || value_depth > c->depths)
        return DAS_ERR_INVALID_ARG;
    const Shape sh = {c->depths, c->layers, c->batch, c->capacity, c->kv_heads, c->head_dim};
    const int slabs = c->depths * c->layers;
    return attention_core(sh, layer, {c->k, false, slabs, (key_depth - 1) * c->layers + layer},
                          {c->v, false, slabs, (value_depth - 1) * c->layers + layer}, prefix_len,
                          block_len, max_block, q, k_blk, v_blk, num_q_heads, softmax_scale, out,
                          lse, workspace, workspace_bytes, clear_status, stream);
}

namespace {

// Depth d of a das_kv_cache_f8: d = R is the bf16 top tensor (slab = layer),
// d < R the e4m3 low tensor (slab (d - 1) * layers + layer).
Operand f8_operand(const das_kv_cache_f8 *c, void *top, void *low, int depth, int layer) {
    if (depth == c->depths) return {top, false, c->layers, layer};
    return {low, true, (c->depths - 1) * c->layers, (depth - 1) * c->layers + layer};
}

das_status attention_f8(const das_kv_cache_f8 *c, int layer, int key_depth, int value_depth,
                        const int32_t *prefix_len, const int32_t *block_len, int max_block,
                        const void *q, const void *k_blk, const void *v_blk, int num_q_heads,
                        float softmax_scale, void *out, float *lse, void *workspace,
                        size_t workspace_bytes, void *stream) {
    if (!cache_f8_ok(c)) {
        if (c && c->head_dim != 64 && c->head_dim != 128) return DAS_ERR_UNSUPPORTED;
        return DAS_ERR_INVALID_ARG;
    }
    if (key_depth < 1 || key_depth > c->depths || value_depth < 1 || value_depth > c->depths ||
        layer < 0 || layer >= c->layers)
        return DAS_ERR_INVALID_ARG;
    const Shape sh = {c->depths, c->layers, c->batch, c->capacity, c->kv_heads, c->head_dim};
    return attention_core(sh, layer, f8_operand(c, c->k_top, c->k_low, key_depth, layer),
                          f8_operand(c, c->v_top, c->v_low, value_depth, layer), prefix_len,
                          block_len, max_block, q, k_blk, v_blk, num_q_heads, softmax_scale, out,
                          lse, workspace, workspace_bytes, false, stream);
}

}  // namespace
}  // namespace das

extern "C" {

size_t das_workspace_size(const das_kv_cache *cache, int num_q_heads, int max_block) {
    if (!cache || cache->kv_heads < 1 || num_q_heads < 1 || num_q_heads % cache->kv_heads != 0 ||
        max_block < 1 || (cache->head_dim != 64 && cache->head_dim != 128))
        return 0;
    const int G = num_q_heads / cache->kv_heads;
    if (max_block > das::kTileKeys || (long long)G * max_block > das::kMaxRows) return 0;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    return das::attn_workspace_bytes(dev, cache->batch, cache->kv_heads, G * max_block,
                                     cache->head_dim);
}

das_status das_mature_v_attention(const das_kv_cache *cache, int layer, int key_depth,
                                  int value_depth, const int32_t *prefix_len,
                                  const int32_t *block_len, int max_block, const void *q,
                                  const void *k_blk, const void *v_blk, int num_q_heads,
                                  float softmax_scale, void *out, float *lse, void *workspace,
                                  size_t workspace_bytes, void *stream) {
    return das::attention(cache, layer, key_depth, value_depth, prefix_len, block_len, max_block,
                          q, k_blk, v_blk, num_q_heads, softmax_scale, out, lse, workspace,
                          workspace_bytes, false, stream);
}

das_status das_verify_attention(const das_kv_cache *cache, int layer, int depth,
                                const int32_t *prefix_len, const int32_t *block_len,
                                int max_block, const void *q, const void *k_blk,
                                const void *v_blk, int num_q_heads, float softmax_scale,
                                void *out, float *lse, void *workspace, size_t workspace_bytes,
                                void *stream) {
    return das::attention(cache, layer, depth, depth, prefix_len, block_len, max_block, q, k_blk,
                          v_blk, num_q_heads, softmax_scale, out, lse, workspace, workspace_bytes,
                          false, stream);
}

das_status das_greedy_accept(const float *logits, const int32_t *draft_ids, int B, int W,
                             int vocab, int32_t *accepted, int32_t *target_ids,
                             int32_t *next_token, void *stream) {
    if (!logits || !draft_ids || !accepted || !target_ids || !next_token || B < 0 || W < 1 ||
        W > 1024 || vocab < 1 || (long long)B * W > 0x7fffffffLL)
        return DAS_ERR_INVALID_ARG;
    return das::accept_launch(logits, draft_ids, B, W, vocab, accepted, target_ids, next_token,
                              static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAS_OK
               : DAS_ERR_CUDA;
}

das_status das_wave_readout(const float *logits, int B, int W, int vocab, int32_t *tokens,
                            int stride, void *stream) {
    if (!logits || !tokens || B < 0 || W < 1 || W > 1024 || vocab < 1 || stride < W + 1 ||
        (long long)B * W > 0x7fffffffLL)
        return DAS_ERR_INVALID_ARG;
    return das::wave_readout_launch(logits, B, W, vocab, tokens, stride,
                                    static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAS_OK
               : DAS_ERR_CUDA;
}

das_status das_kv_append(const das_kv_cache *cache, const void *k_new, const void *v_new,
                         const int32_t *accepted, int W, int32_t *prefix_len,
                         int32_t *error_flag, void *stream) {
    if (!das::cache_ok(cache) || !k_new || !v_new || !accepted || !prefix_len || !error_flag ||
        W < 1 || W > cache->capacity || !das::aligned16(k_new) || !das::aligned16(v_new))
        return DAS_ERR_INVALID_ARG;
    return das::append_launch(*cache, k_new, v_new, accepted, W, prefix_len, error_flag,
                              static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAS_OK
               : DAS_ERR_CUDA;
}

size_t das_workspace_size_f8(const das_kv_cache_f8 *cache, int num_q_heads, int max_block) {
    if (!cache) return 0;
    das_kv_cache view = {cache->k_top, cache->v_top, cache->depths, cache->layers, cache->batch,
                         cache->capacity, cache->kv_heads, cache->head_dim};
    return das_workspace_size(&view, num_q_heads, max_block);
}

das_status das_mature_v_attention_f8(const das_kv_cache_f8 *cache, int layer, int key_depth,
                                     int value_depth, const int32_t *prefix_len,
                                     const int32_t *block_len, int max_block, const void *q,
                                     const void *k_blk, const void *v_blk, int num_q_heads,
                                     float softmax_scale, void *out, float *lse, void *workspace,
                                     size_t workspace_bytes, void *stream) {
    return das::attention_f8(cache, layer, key_depth, value_depth, prefix_len, block_len,
                             max_block, q, k_blk, v_blk, num_q_heads, softmax_scale, out, lse,
                             workspace, workspace_bytes, stream);
}

das_status das_kv_append_f8(const das_kv_cache_f8 *cache, const void *k_new, const void *v_new,
                            const int32_t *accepted, int W, int32_t *prefix_len,
                            int32_t *error_flag, void *stream) {
    if (!das::cache_f8_ok(cache) || !k_new || !v_new || !accepted || !prefix_len || !error_flag ||
        W < 1 || W > cache->capacity || !das::aligned16(k_new) || !das::aligned16(v_new))
        return DAS_ERR_INVALID_ARG;
    return das::append_f8_launch(*cache, k_new, v_new, accepted, W, prefix_len, error_flag,
                                 static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? DAS_OK
               : DAS_ERR_CUDA;
}

const char *das_status_string(das_status s) {
    switch (s) {
        case DAS_OK: return "ok";
        case DAS_ERR_INVALID_ARG: return "invalid argument";
        case DAS_ERR_UNSUPPORTED: return "unsupported shape";
        case DAS_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case DAS_ERR_CUDA: return "CUDA runtime error";
    }
    return "unknown status";
}

}  // extern "C"
