/*
 * das.h -- C ABI of the GB300 (sm_103a) library for the data-parallel hot path
 * of DAS-Wave decoding ("Shallow Queries, Mature Values: Depth-Asynchronous
 * Self-Speculation for Looped Transformers").
 *
 * The library computes, on one GPU:
 *   das_mature_v_attention  depth-asynchronous draft attention, Eqs. 2-3
 *                           (Sec. 3.2), with explicit read depths (Eq. 4):
 *                           Mature-V is (key_depth, value_depth) = (r, R);
 *   das_verify_attention    the full-depth verify attention of Sec. 3.4
 *                           (Eq. 7): the same with key and value depth equal;
 *   das_greedy_accept       greedy acceptance of Sec. 3.4;
 *   das_kv_append           the commit of Sec. 3.4 / App. B.1.
 *
 * Conventions shared by every entry point
 *   - Every pointer argument marked "device" is device memory owned by the
 *     caller; the library never allocates or frees device memory.  Host
 *     pointers are read during the call only.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; 0 = legacy default
 *     stream) and never synchronise the host.  Errors found on the host
 *     (arguments) are returned before anything is launched and nothing is
 *     written.  Errors found on the device are reported through flags
 *     described at each call.
 *   - bf16 tensors are IEEE bfloat16, row-major in the stated index order,
 *     densely packed, with base addresses aligned to 16 bytes.
 *   - Recurrent depths are numbered as in the paper: 1..R, R = full depth.
 *     Depth d is stored in slab d-1 of the cache.
 *   - Query head h reads kv head h / G, G = num_q_heads / kv_heads
 *     (contiguous grouping; the paper does not fix one).
 */
#ifndef DAS_H
#define DAS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DAS_OK = 0,
    DAS_ERR_INVALID_ARG = 1, /* a null pointer, bad size, depth or alignment */
    DAS_ERR_UNSUPPORTED = 2, /* a shape outside what the kernels implement  */
    DAS_ERR_WORKSPACE = 3,   /* workspace missing or smaller than required  */
    DAS_ERR_CUDA = 4         /* a CUDA runtime call failed                  */
} das_status;

/*
 * Depth-indexed KV cache of the verified prefix (Sec. 2: the cache holds
 * K_C^{r,l} and V_C^{r,l} for every recurrent depth r and core layer l; only
 * target-materialized positions are stored, App. B.1).
 *   k, v   device bf16 [depths][layers][batch][capacity][kv_heads][head_dim]
 * Slab (d, l, b) is contiguous, so the keys of one depth and the values of
 * another stream independently.  Positions >= prefix_len[b] may hold anything.
 */
typedef struct {
    void *k;
    void *v;
    int depths;   /* R, number of stored recurrent depths, 1..63        */
    int layers;   /* core layers                                        */
    int batch;    /* sequences                                          */
    int capacity; /* positions per sequence                             */
    int kv_heads; /* Hkv                                                */
    int head_dim; /* D: 64 or 128                                       */
} das_kv_cache;

/*
 * Bytes of device workspace that das_mature_v_attention and
 * das_verify_attention need for this cache shape, num_q_heads and max_block
 * on the current device.  Returns 0 for shapes the kernels do not support.
 * The first 256 bytes of a workspace are a header; its first int32 is a
 * status word that the kernels OR with 1 if an internal wait ran out (a bug
 * guard; it stays set until the caller clears it).  Zero a new workspace once
 * before its first use.
 */
size_t das_workspace_size(const das_kv_cache *cache, int num_q_heads, int max_block);

/*
 * Depth-asynchronous attention, Eqs. 2-3 (Sec. 3.2).  For each sequence b,
 * query head h and block row i < block_len[b]:
 *   keys   = [ K[key_depth][layer][b][j][h/G]   for j < prefix_len[b] ]
 *            ++ [ k_blk[b][j][h/G] for j <= i ]      (causal mask M)
 *   values = [ V[value_depth][layer][b][j][h/G] for j < prefix_len[b] ]
 *            ++ [ v_blk[b][j][h/G] for j <= i ]
 *   s_j = softmax_scale * <q[b][i][h], keys_j>,  one softmax over all j,
 *   out[b][i][h] = sum_j softmax(s)_j values_j,
 *   lse[b][h][i] = ln sum_j exp(s_j).
 * Mature-V for a draft at depth r is (key_depth, value_depth) = (r, R);
 * Aligned (r, r), Deep K (R, r) and Deep K/V (R, R) are the other policies
 * of Eq. 4.  The block's own K/V (k_blk, v_blk) are produced by the current
 * draft and are never written to the cache by this call (Sec. 3.2, 3.3).
 *
 *   cache          the depth-indexed cache (read only)
 *   layer          core layer, 0 <= layer < cache->layers
 *   key_depth      kappa, 1..cache->depths
 *   value_depth    nu, 1..cache->depths
 *   prefix_len     device int32 [batch]: verified prefix length per sequence,
 *                  0..capacity
 *   block_len      device int32 [batch]: draft rows per sequence, 0..max_block
 *   max_block      rows allocated per sequence in q/k_blk/v_blk/out/lse;
 *                  (num_q_heads / kv_heads) * max_block <= 64, max_block <= 64
 *   q              device bf16 [batch][max_block][num_q_heads][head_dim]
 *   k_blk, v_blk   device bf16 [batch][max_block][kv_heads][head_dim]
 *   num_q_heads    Hq, a multiple of kv_heads
 *   softmax_scale  scale of Eq. 2; <= 0 selects 1/sqrt(head_dim)
 *   out            device bf16 [batch][max_block][num_q_heads][head_dim];
 *                  rows i >= block_len[b] are written as 0
 *   lse            device fp32 [batch][num_q_heads][max_block]; -inf for rows
 *                  i >= block_len[b]
 *   workspace      device scratch of at least das_workspace_size() bytes,
 *                  aligned to 256 bytes; calls sharing a workspace must not
 *                  overlap in time
 * Device-side: prefix_len or block_len outside their ranges are clamped and
 * bit 1 of the workspace status word is set.
 */
das_status das_mature_v_attention(const das_kv_cache *cache, int layer, int key_depth,
                                  int value_depth, const int32_t *prefix_len,
                                  const int32_t *block_len, int max_block, const void *q,
                                  const void *k_blk, const void *v_blk, int num_q_heads,
                                  float softmax_scale, void *out, float *lse, void *workspace,
                                  size_t workspace_bytes, void *stream);

/*
 * Independent full-depth verify attention (Sec. 3.4, Eq. 7): the verifier
 * input [x_t, y_1 .. y_{w-1}] is the block (block_len[b] = w rows), it
 * attends to the verified prefix at one depth for keys and values alike
 * (depth = R for the target's last recurrence; every depth d of the verify
 * pass uses the same call) and to itself under the causal mask.  Arguments
 * and results as das_mature_v_attention with key_depth = value_depth = depth.
 */
das_status das_verify_attention(const das_kv_cache *cache, int layer, int depth,
                                const int32_t *prefix_len, const int32_t *block_len,
                                int max_block, const void *q, const void *k_blk,
                                const void *v_blk, int num_q_heads, float softmax_scale,
                                void *out, float *lse, void *workspace, size_t workspace_bytes,
                                void *stream);

/*
 * Greedy acceptance (Sec. 3.4).  logits[b][i] stands for the verifier's
 * conditional p_{i+1} of proposal y_{i+1} = draft_ids[b][i]:
 *   target_ids[b][i] = argmax_v logits[b][i][v]   (smallest index on ties;
 *                      binary32 comparisons; NaN logits are out of contract)
 *   accepted[b]      = number of leading i with draft_ids[b][i] == target_ids[b][i]
 *   next_token[b]    = target_ids[b][accepted[b]] if accepted[b] < W (the target
 *                      prediction emitted at the first mismatch), otherwise
 *                      draft_ids[b][W-1] (every proposal accepted: no further
 *                      conditional exists, and the last accepted token becomes
 *                      the next anchor).
 *   logits      device fp32 [B][W][vocab]
 *   draft_ids   device int32 [B][W]
 *   accepted    device int32 [B];  target_ids device int32 [B][W];
 *   next_token  device int32 [B]
 * Requires 1 <= W <= 1024, 1 <= vocab < 2^31.
 */
das_status das_greedy_accept(const float *logits, const int32_t *draft_ids, int B, int W,
                             int vocab, int32_t *accepted, int32_t *target_ids,
                             int32_t *next_token, void *stream);

/*
 * Shifted token readout of a DAS-Wave refinement round (Sec. 3.3, Eq. 6).
 * After the k recurrent draft updates of round j over the W = W_j active
 * positions [x_t, z_1 .. z_{W-1}] (W_j = min(gamma, W_init + j), Eq. 5), the
 * readout of position i updates the guess of the following position:
 *   tokens[b][i + 1] = argmax_v logits[b][i][v]   for 0 <= i < W
 * (smallest index on ties, binary32 comparisons, as das_greedy_accept).
 * tokens[b][0] (the anchor) and tokens[b][i] for i > W are not written; the
 * readout of the last active position is the candidate that enters the
 * window in the next round.
 *   logits   device fp32 [B][W][vocab]
 *   tokens   device int32 [B][stride], stride >= W + 1
 * Requires 1 <= W <= 1024, 1 <= vocab < 2^31.
 */
das_status das_wave_readout(const float *logits, int B, int W, int vocab, int32_t *tokens,
                            int stride, void *stream);

/*
 * Commit (Sec. 3.4; App. B.1): the verifier consumed W inputs
 * [x_t, y_1 .. y_{W-1}] and produced their K/V at every depth and layer.
 * With accepted[b] = a proposals accepted, the first n = min(a + 1, W) inputs
 * (the anchor and the accepted proposals that were verifier inputs) are
 * materialized: their staged K/V are copied byte for byte to cache positions
 * prefix_len[b] .. prefix_len[b] + n - 1 at every depth and layer, and
 * prefix_len[b] += n.  Rejected candidates' K/V are discarded.
 *   k_new, v_new  device bf16 [depths][layers][batch][W][kv_heads][head_dim]
 *   accepted      device int32 [batch] (as written by das_greedy_accept)
 *   prefix_len    device int32 [batch], updated in place
 *   error_flag    device int32: set to 1 (never cleared) if a sequence would
 *                 exceed the capacity; that sequence's cache and prefix_len
 *                 are left untouched
 * Requires 1 <= W <= capacity.
 */
das_status das_kv_append(const das_kv_cache *cache, const void *k_new, const void *v_new,
                         const int32_t *accepted, int W, int32_t *prefix_len,
                         int32_t *error_flag, void *stream);

/*
 * Bytes of device scratch built into the library for
 * das_mature_v_attention_noalloc (32 MiB on every device that loads it).
 */
#define DAS_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

/*
 * das_mature_v_attention without a caller-provided workspace.  The paper has
 * no counterpart: this is for callers that cannot allocate device memory when
 * they call (a fixed memory plan in a serving loop, a plugin that only
 * receives the tensors it works on, a host that forbids cudaMalloc after
 * start-up).  The split-K scratch is a fixed array of
 * DAS_NOALLOC_SCRATCH_BYTES inside the library's device image, present on
 * every device that loads the library until the process exits; this call
 * allocates nothing and calls no allocating routine.
 *   - Arguments and results as das_mature_v_attention, minus the workspace.
 *   - Returns DAS_ERR_WORKSPACE if the shape needs more scratch than
 *     DAS_NOALLOC_SCRATCH_BYTES (das_workspace_size() tells how much), with
 *     nothing launched.
 *   - The first call on a device looks up the array's device address (set-up
 *     done once per device, then kept); make that first call before any CUDA
 *     graph capture on that device.  After cudaDeviceReset on a device, later
 *     calls in that process are invalid.
 *   - All calls share the array and it keeps the last call's contents: calls
 *     that overlap in time on the GPU race and must be ordered by the caller.
 *     A call that passes its argument checks clears the status word at the
 *     array's head (on `stream`, just before its kernels); its bits, as for
 *     the workspace status word of das_mature_v_attention, are read with
 *     das_noalloc_status until the next call.  A call that returns an error
 *     enqueues nothing.
 */
das_status das_mature_v_attention_noalloc(const das_kv_cache *cache, int layer, int key_depth,
                                          int value_depth, const int32_t *prefix_len,
                                          const int32_t *block_len, int max_block, const void *q,
                                          const void *k_blk, const void *v_blk, int num_q_heads,
                                          float softmax_scale, void *out, float *lse,
                                          void *stream);

/*
 * Copies the status word of das_mature_v_attention_noalloc's scratch on the
 * current device (bit 0: an internal wait timed out; bit 1: a prefix or block
 * length was out of range and clamped) to `dst` (host or device memory,
 * 4 bytes) on `stream`, after the work enqueued there before it.  Allocates
 * nothing.  The paper has no counterpart.
 */
das_status das_noalloc_status(int32_t *dst, void *stream);

/*
 * A depth-indexed cache whose depths below R are stored as 8-bit floats.
 * The paper has no counterpart: it keeps every depth in the model's precision.
 * This variant halves the bytes of the shallow-depth stream that Mature-V
 * reads (keys at depth r < R) while the mature depth R that carries the
 * values and the verifier's reads at R stays bf16.
 *   k_top, v_top  device bf16 [layers][batch][capacity][kv_heads][head_dim]:
 *                 depth R
 *   k_low, v_low  device e4m3 (OCP FP8 E4M3: 1 sign, 4 exponent bits with
 *                 bias 7, 3 mantissa bits; no infinities, S.1111.111 is NaN;
 *                 largest finite 448)
 *                 [depths - 1][layers][batch][capacity][kv_heads][head_dim]:
 *                 depth d < R at slab d - 1; may be NULL when depths == 1
 * All pointers 16-byte aligned; the caller owns the memory.
 */
typedef struct {
    void *k_top;
    void *v_top;
    void *k_low;
    void *v_low;
    int depths, layers, batch, capacity, kv_heads, head_dim;
} das_kv_cache_f8;

/* Workspace bytes for das_mature_v_attention_f8 (as das_workspace_size). */
size_t das_workspace_size_f8(const das_kv_cache_f8 *cache, int num_q_heads, int max_block);

/*
 * das_mature_v_attention over a das_kv_cache_f8: keys are read at key_depth
 * and values at value_depth from k_top / v_top (depth R) or from k_low / v_low
 * (depths below R, e4m3), so Eqs. 2-3 are evaluated on the stored values.
 * key_depth = value_depth = d is the verify attention of depth d (Sec. 3.4).
 * All other arguments, results and limits as das_mature_v_attention.
 * e4m3 operands are widened exactly to bf16 before the products, except for
 * e4m3 keys with bf16 values at head_dim 128 (Mature-V, key_depth < R =
 * value_depth): there the scores are e4m3 products of the stored keys with
 * each query row split exactly into two e4m3 parts under a power of two per
 * row (exact for elements down to about 2^-9 of the row's largest magnitude,
 * fp32 accumulation), and the queries must be finite.
 */
das_status das_mature_v_attention_f8(const das_kv_cache_f8 *cache, int layer, int key_depth,
                                     int value_depth, const int32_t *prefix_len,
                                     const int32_t *block_len, int max_block, const void *q,
                                     const void *k_blk, const void *v_blk, int num_q_heads,
                                     float softmax_scale, void *out, float *lse, void *workspace,
                                     size_t workspace_bytes, void *stream);

/*
 * das_kv_append into a das_kv_cache_f8: the staged bf16 K/V of depth R are
 * copied byte for byte; those of depths below R are rounded to e4m3 (round to
 * nearest, ties to even; magnitudes above 448 saturate to 448; NaN stays NaN).
 * Arguments and errors as das_kv_append.
 */
das_status das_kv_append_f8(const das_kv_cache_f8 *cache, const void *k_new, const void *v_new,
                            const int32_t *accepted, int W, int32_t *prefix_len,
                            int32_t *error_flag, void *stream);

/* Static text for a status code. */
const char *das_status_string(das_status s);

#ifdef __cplusplus
}
#endif

#endif /* DAS_H */
