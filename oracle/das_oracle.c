/*
 * das_oracle.c -- plain, slow, fp64 CPU oracle for the DAS-Wave hot path
 * ("Shallow Queries, Mature Values: Depth-Asynchronous Self-Speculation for
 * Looped Transformers").
 *
 * TEST INFRASTRUCTURE ONLY.  This file checks the CUDA library; it is not part
 * of it.  Only the test suite, the smoke check and the benchmark's CPU-baseline
 * leg may load it.  It shares no code, header, table or helper with the CUDA
 * path, and the CUDA path never calls it.
 *
 * What it computes, each function written straight from the paper:
 *
 *   das_oracle_attend_seq   depth-asynchronous attention for one sequence and
 *                           one core layer, Eqs. 2-3 (Sec. 3.2): one softmax
 *                           over [prefix keys read at depth kappa ; the draft
 *                           block's own keys] under the causal mask M, output
 *                           = weights times [prefix values read at depth nu ;
 *                           block values].
 *   das_oracle_attention    the same over a whole depth-indexed cache
 *                           [depth][layer][batch][token][kv_head][head_dim];
 *                           selects the key slab at depth kappa and the value
 *                           slab at depth nu (read policies, Eq. 4).  With
 *                           kappa = nu = R it is the full-depth verify
 *                           attention of Sec. 3.4 (Eq. 7).
 *   das_oracle_greedy_accept greedy acceptance of Sec. 3.4.
 *   das_oracle_wave_readout  the shifted token readout of a DAS-Wave
 *                           refinement round, Eq. 6 (Sec. 3.3).
 *   das_oracle_e4m3_*        the 8-bit storage of depths below R used by the
 *                           library's e4m3 cache variant (not in the paper):
 *                           exact decoding, and rounding to nearest-even
 *                           with saturation at +-448, from the format's
 *                           definition (OCP FP8 E4M3: bias 7, 3 mantissa
 *                           bits, no infinities, S.1111.111 = NaN).
 *   das_oracle_kv_append     the commit of Sec. 3.4 / App. B.1: keep the K/V of
 *                           accepted, materialized verifier inputs at every
 *                           depth and layer.
 *
 * Readings where the paper is silent (each restated where it is used):
 *   - depths are numbered 1..R as in the paper; depth d lives at slab d-1;
 *   - query head h uses kv head floor(h / G), G = Hq / Hkv (contiguous groups);
 *   - block row i sees every prefix key and block keys j <= i;
 *   - lse is the natural log of the softmax denominator over the scaled scores;
 *   - argmax ties go to the smallest vocabulary index;
 *   - a sequence with a accepted proposals out of w materializes
 *     n = min(a + 1, w) verifier inputs [x_t, y_1 .. y_{n-1}].
 *
 * Arithmetic: every bf16 input is widened exactly to double; dot products,
 * max, exp, sums and the weighted value sum are done in double in the order
 * the definition states (keys in position order).  No blocking, no online
 * rescaling, no fusion.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* bf16 is the upper half of an IEEE binary32; widening is exact. */
static double bf16_to_double(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * Attention of Eqs. 2-3 for one sequence at one core layer.
 *
 *   q      [T][Hq][D]   queries of the draft block (rows i < block_len used)
 *   k_pre  [P][Hkv][D]  verified-prefix keys, already the depth-kappa slab
 *   v_pre  [P][Hkv][D]  verified-prefix values, already the depth-nu slab
 *   k_blk  [T][Hkv][D]  the block's own keys (produced by the current draft)
 *   v_blk  [T][Hkv][D]  the block's own values
 *   prefix_lo, prefix_hi  prefix positions [lo, hi) that take part (the whole
 *                         prefix is [0, P); a sub-range gives the partial
 *                         result over that chunk only)
 *   use_block            1: block keys j <= i take part (causal mask M);
 *                        0: prefix keys only
 *   scale                softmax scale; Eq. 2 uses 1/sqrt(d_h)
 *   out    [T][Hq][D]   double; rows i >= block_len, or rows that see no key,
 *                        are 0
 *   lse    [Hq][T]      double, natural log of sum_j exp(s_j); -inf where a
 *                        row sees no key
 *   h_lo, h_hi           query heads [h_lo, h_hi) to compute (others untouched)
 */
void das_oracle_attend_seq(int P, int T, int block_len, int Hq, int Hkv, int D,
                           const uint16_t *q, const uint16_t *k_pre,
                           const uint16_t *v_pre, const uint16_t *k_blk,
                           const uint16_t *v_blk, int prefix_lo, int prefix_hi,
                           int use_block, double scale, double *out,
                           double *lse, int h_lo, int h_hi) {
    int G = Hq / Hkv;
    int max_keys = (prefix_hi > prefix_lo ? prefix_hi - prefix_lo : 0) + T;
    double *s = (double *)malloc(sizeof(double) * (size_t)(max_keys > 0 ? max_keys : 1));
    double *qd = (double *)malloc(sizeof(double) * (size_t)D);
    for (int h = h_lo; h < h_hi; ++h) {
        int hk = h / G; /* contiguous GQA grouping */
        for (int i = 0; i < T; ++i) {
            double *o = out + ((size_t)i * Hq + h) * D;
            for (int d = 0; d < D; ++d) o[d] = 0.0;
            lse[(size_t)h * T + i] = -INFINITY;
            if (i >= block_len) continue;
            for (int d = 0; d < D; ++d)
                qd[d] = bf16_to_double(q[((size_t)i * Hq + h) * D + d]);

            /* Scores over the concatenated key list [K_C^kappa ; K_U^cur]:
             * prefix positions lo..hi-1, then block positions 0..i (mask M). */
            int n = 0;
            for (int j = prefix_lo; j < prefix_hi; ++j) {
                const uint16_t *kr = k_pre + ((size_t)j * Hkv + hk) * D;
                double dot = 0.0;
                for (int d = 0; d < D; ++d) dot += qd[d] * bf16_to_double(kr[d]);
                s[n++] = dot * scale;
            }
            int nblk = 0;
            if (use_block) {
                for (int j = 0; j <= i; ++j) {
                    const uint16_t *kr = k_blk + ((size_t)j * Hkv + hk) * D;
                    double dot = 0.0;
                    for (int d = 0; d < D; ++d) dot += qd[d] * bf16_to_double(kr[d]);
                    s[n++] = dot * scale;
                }
                nblk = i + 1;
            }
            if (n == 0) continue;

            /* softmax: m = max_j s_j, Z = sum_j exp(s_j - m), lse = m + ln Z */
            double m = s[0];
            for (int j = 1; j < n; ++j)
                if (s[j] > m) m = s[j];
            double Z = 0.0;
            for (int j = 0; j < n; ++j) Z += exp(s[j] - m);
            double l = m + log(Z);
            lse[(size_t)h * T + i] = l;

            /* Eq. 3: O = Pi_C V_C^nu + Pi_U V_U^cur */
            int t = 0;
            for (int j = prefix_lo; j < prefix_hi; ++j, ++t) {
                double p = exp(s[t] - l);
                const uint16_t *vr = v_pre + ((size_t)j * Hkv + hk) * D;
                for (int d = 0; d < D; ++d) o[d] += p * bf16_to_double(vr[d]);
            }
            for (int j = 0; j < nblk; ++j, ++t) {
                double p = exp(s[t] - l);
                const uint16_t *vr = v_blk + ((size_t)j * Hkv + hk) * D;
                for (int d = 0; d < D; ++d) o[d] += p * bf16_to_double(vr[d]);
            }
        }
    }
    free(qd);
    free(s);
}

/* ---------------------------------------------------------------------------
 * Whole-cache form.  The cache is [depths][layers][batch][capacity][Hkv][D]
 * bf16; recurrent depth d (1..depths) is slab d-1.  For sequence b the key
 * slab is K[kappa-1][layer][b] and the value slab V[nu-1][layer][b], each
 * [capacity][Hkv][D] of which the first prefix_len[b] tokens are the verified
 * prefix C.  Work is spread over (sequence, query head) with plain threads.
 * ------------------------------------------------------------------------- */
typedef struct {
    const uint16_t *k_cache, *v_cache;
    int depths, layers, batch, capacity, Hkv, D;
    int layer, key_depth, value_depth;
    const int32_t *prefix_len, *block_len;
    int max_block;
    const uint16_t *q, *k_blk, *v_blk;
    int Hq;
    double scale;
    int use_block;
    double *out, *lse;
    int next; /* next (b, h) work item */
    pthread_mutex_t mu;
} attn_job;

static void *attn_worker(void *arg) {
    attn_job *J = (attn_job *)arg;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        int item = J->next++;
        pthread_mutex_unlock(&J->mu);
        if (item >= J->batch * J->Hq) break;
        int b = item / J->Hq, h = item % J->Hq;
        size_t slab = (size_t)J->capacity * J->Hkv * J->D;
        const uint16_t *ks =
            J->k_cache + (((size_t)(J->key_depth - 1) * J->layers + J->layer) * J->batch + b) * slab;
        const uint16_t *vs =
            J->v_cache + (((size_t)(J->value_depth - 1) * J->layers + J->layer) * J->batch + b) * slab;
        size_t qrow = (size_t)J->max_block * J->Hq * J->D;
        size_t kvrow = (size_t)J->max_block * J->Hkv * J->D;
        das_oracle_attend_seq(J->prefix_len[b], J->max_block, J->block_len[b], J->Hq,
                              J->Hkv, J->D, J->q + b * qrow, ks, vs,
                              J->k_blk + b * kvrow, J->v_blk + b * kvrow, 0,
                              J->prefix_len[b], J->use_block, J->scale,
                              J->out + b * qrow, J->lse + (size_t)b * J->Hq * J->max_block,
                              h, h + 1);
    }
    return NULL;
}

/*
 * Returns 0 on success, 1 on an argument the definition does not cover.
 *   q      [batch][max_block][Hq][D] bf16;  k_blk, v_blk [batch][max_block][Hkv][D]
 *   out    [batch][max_block][Hq][D] double; lse [batch][Hq][max_block] double
 *   scale <= 0 selects 1/sqrt(D) (Eq. 2).
 */
int das_oracle_attention(const uint16_t *k_cache, const uint16_t *v_cache, int depths,
                         int layers, int batch, int capacity, int Hkv, int D, int layer,
                         int key_depth, int value_depth, const int32_t *prefix_len,
                         const int32_t *block_len, int max_block, const uint16_t *q,
                         const uint16_t *k_blk, const uint16_t *v_blk, int Hq, double scale,
                         int use_block, double *out, double *lse, int nthreads) {
    if (Hkv <= 0 || Hq % Hkv != 0 || key_depth < 1 || key_depth > depths ||
        value_depth < 1 || value_depth > depths || layer < 0 || layer >= layers)
        return 1;
    for (int b = 0; b < batch; ++b)
        if (prefix_len[b] < 0 || prefix_len[b] > capacity || block_len[b] < 0 ||
            block_len[b] > max_block)
            return 1;
    attn_job J;
    J.k_cache = k_cache; J.v_cache = v_cache;
    J.depths = depths; J.layers = layers; J.batch = batch; J.capacity = capacity;
    J.Hkv = Hkv; J.D = D; J.layer = layer; J.key_depth = key_depth;
    J.value_depth = value_depth; J.prefix_len = prefix_len; J.block_len = block_len;
    J.max_block = max_block; J.q = q; J.k_blk = k_blk; J.v_blk = v_blk; J.Hq = Hq;
    J.scale = scale > 0.0 ? scale : 1.0 / sqrt((double)D);
    J.use_block = use_block; J.out = out; J.lse = lse; J.next = 0;
    pthread_mutex_init(&J.mu, NULL);
    if (nthreads < 1) nthreads = 1;
    pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
    int started = 0;
    for (int t = 1; t < nthreads; ++t)
        if (pthread_create(&th[started], NULL, attn_worker, &J) == 0) ++started;
    attn_worker(&J);
    for (int t = 0; t < started; ++t) pthread_join(th[t], NULL);
    free(th);
    pthread_mutex_destroy(&J.mu);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Greedy acceptance (Sec. 3.4).  For sequence b the verifier returns
 * conditionals p_1..p_w; here logits[b][i-1][:] stands for p_i.
 *   yhat_i = argmax_v p_i(v)            (ties: smallest index)
 *   proposals y_i = draft[b][i-1] are accepted in order while y_i == yhat_i;
 *   a_b = number accepted;
 *   next_token[b] = yhat_{a_b+1} when a_b < w (the target prediction emitted
 *   at the first mismatch), else y_w: with every proposal accepted (m = w) no
 *   extra conditional is left, and the last accepted token becomes the next
 *   anchor.
 * target_ids[b][i] = yhat_{i+1} for every i.  Logits are compared in their
 * own precision (binary32), exactly.
 * ------------------------------------------------------------------------- */
void das_oracle_greedy_accept(const float *logits, const int32_t *draft, int B, int W,
                              int vocab, int32_t *accepted, int32_t *target_ids,
                              int32_t *next_token) {
    for (int b = 0; b < B; ++b) {
        for (int i = 0; i < W; ++i) {
            const float *row = logits + ((size_t)b * W + i) * vocab;
            int best = 0;
            for (int v = 1; v < vocab; ++v)
                if (row[v] > row[best]) best = v; /* strict: first maximum wins */
            target_ids[b * W + i] = best;
        }
        int a = 0;
        while (a < W && draft[b * W + a] == target_ids[b * W + a]) ++a;
        accepted[b] = a;
        next_token[b] = a < W ? target_ids[b * W + a] : draft[b * W + W - 1];
    }
}

/* ---------------------------------------------------------------------------
 * Shifted readout of a DAS-Wave refinement round (Sec. 3.3, Eq. 6).  After the
 * k recurrent draft updates of round j over the W_j active positions
 * [x_t, z_1 .. z_{W_j - 1}], the readout of position i updates the guess of
 * the following position: z_{i+1} = argmax_v logits[b][i][v] for 0 <= i < W.
 * tokens is [B][stride] with stride >= W + 1; position 0 (the anchor) and
 * positions past W are left as they are.  First maximum on ties, binary32
 * comparisons, as in greedy acceptance.
 * ------------------------------------------------------------------------- */
void das_oracle_wave_readout(const float *logits, int B, int W, int vocab, int32_t *tokens,
                             int stride) {
    for (int b = 0; b < B; ++b)
        for (int i = 0; i < W; ++i) {
            const float *row = logits + ((size_t)b * W + i) * vocab;
            int best = 0;
            for (int v = 1; v < vocab; ++v)
                if (row[v] > row[best]) best = v;
            tokens[(size_t)b * stride + i + 1] = best;
        }
}

/* ---------------------------------------------------------------------------
 * e4m3 (OCP FP8 E4M3): sign s, exponent field e (4 bits, bias 7), mantissa m
 * (3 bits).  e = 0: (-1)^s m/8 2^-6; otherwise (-1)^s (1 + m/8) 2^(e-7);
 * e = 15, m = 7 is NaN (no infinities); the largest finite value is 448.
 * ------------------------------------------------------------------------- */
double das_oracle_e4m3_decode(uint8_t c) {
    const int s = c >> 7, e = (c >> 3) & 15, m = c & 7;
    if (e == 15 && m == 7) return NAN;
    const double mag = e == 0 ? ldexp((double)m / 8.0, -6) : ldexp(1.0 + m / 8.0, e - 7);
    return s ? -mag : mag;
}

/* Nearest e4m3 value, ties to the even mantissa; magnitudes above 448 and
 * infinities become +-448; NaN becomes 0x7F. */
uint8_t das_oracle_e4m3_encode(double x) {
    if (isnan(x)) return 0x7F;
    const uint8_t s = signbit(x) ? 0x80 : 0x00;
    const double a = fabs(x);
    if (a > 448.0) return s | 0x7E;
    if (a < ldexp(1.0, -6)) {                 /* subnormal range: steps of 2^-9 */
        const double q = nearbyint(ldexp(a, 9));  /* current mode: to nearest, ties even */
        return s | (uint8_t)q;                /* q = 8 is the smallest normal, 0x08 */
    }
    int E;
    frexp(a, &E);                             /* a = f 2^E, f in [0.5, 1) */
    E -= 1;                                   /* a = (1 + t) 2^E, t in [0, 1) */
    double q = nearbyint(ldexp(a, 3 - E));    /* 8 (1 + t), in [8, 16] */
    if (q == 16.0) {                          /* rounded up to the next binade */
        q = 8.0;
        E += 1;
    }
    const int e = E + 7, m = (int)q - 8;
    if (e > 15 || (e == 15 && m == 7)) return s | 0x7E;
    return s | (uint8_t)(e << 3) | (uint8_t)m;
}

void das_oracle_e4m3_decode_n(const uint8_t *in, double *out, size_t n) {
    for (size_t i = 0; i < n; ++i) out[i] = das_oracle_e4m3_decode(in[i]);
}

/* bf16 bits -> e4m3 codes (every bf16 value is exact in double). */
void das_oracle_e4m3_from_bf16_n(const uint16_t *in, uint8_t *out, size_t n) {
    for (size_t i = 0; i < n; ++i) {
        union { uint32_t u; float f; } v;
        v.u = (uint32_t)in[i] << 16;
        out[i] = das_oracle_e4m3_encode((double)v.f);
    }
}

/* ---------------------------------------------------------------------------
 * Commit (Sec. 3.4, App. B.1).  The verifier consumed [x_t, y_1 .. y_{w-1}]
 * and produced their K/V at every depth and core layer, staged as
 * k_new/v_new [depths][layers][batch][w][Hkv][D].  With a_b proposals
 * accepted, the materialized inputs to keep are the first n_b = min(a_b+1, w)
 * of them (the anchor plus the accepted proposals that were verifier inputs);
 * the rest are discarded.  They are copied, byte for byte, to cache positions
 * prefix_len[b] .. prefix_len[b]+n_b-1 at every depth and layer, and
 * prefix_len[b] grows by n_b.  A sequence whose new length would exceed the
 * capacity is left untouched and *error_flag is set to 1.
 * ------------------------------------------------------------------------- */
void das_oracle_kv_append(uint16_t *k_cache, uint16_t *v_cache, int depths, int layers,
                          int batch, int capacity, int Hkv, int D, const uint16_t *k_new,
                          const uint16_t *v_new, const int32_t *accepted, int W,
                          int32_t *prefix_len, int32_t *error_flag) {
    size_t row = (size_t)Hkv * D;
    for (int b = 0; b < batch; ++b) {
        int a = accepted[b];
        if (a < 0) a = 0;
        int n = a + 1 < W ? a + 1 : W;
        int p = prefix_len[b];
        if (p + n > capacity) {
            *error_flag = 1;
            continue;
        }
        for (int d = 0; d < depths; ++d)
            for (int l = 0; l < layers; ++l) {
                size_t cs = (((size_t)d * layers + l) * batch + b) * capacity;
                size_t ss = (((size_t)d * layers + l) * batch + b) * W;
                memcpy(k_cache + (cs + p) * row, k_new + ss * row, sizeof(uint16_t) * n * row);
                memcpy(v_cache + (cs + p) * row, v_new + ss * row, sizeof(uint16_t) * n * row);
            }
        prefix_len[b] = p + n;
    }
}


/* ---------------------------------------------------------------------------
 * The commit into an e4m3 cache (the library's variant, not in the paper):
 * as das_oracle_kv_append over k_new/v_new [R][L][B][W][Hkv][D] (bf16), with
 * depth R copied into k_top/v_top [L][B][cap][Hkv][D] (bf16) and depths
 * d < R rounded (das_oracle_e4m3_encode) into k_low/v_low
 * [R-1][L][B][cap][Hkv][D] (e4m3).
 * ------------------------------------------------------------------------- */
void das_oracle_kv_append_f8(uint16_t *k_top, uint16_t *v_top, uint8_t *k_low, uint8_t *v_low,
                             int depths, int layers, int batch, int capacity, int Hkv, int D,
                             const uint16_t *k_new, const uint16_t *v_new, const int32_t *accepted,
                             int W, int32_t *prefix_len, int32_t *error_flag) {
    size_t row = (size_t)Hkv * D;
    for (int b = 0; b < batch; ++b) {
        int a = accepted[b];
        if (a < 0) a = 0;
        int n = a + 1 < W ? a + 1 : W;
        int p = prefix_len[b];
        if (p + n > capacity) {
            *error_flag = 1;
            continue;
        }
        for (int d = 0; d < depths; ++d)
            for (int l = 0; l < layers; ++l) {
                size_t ss = (((size_t)d * layers + l) * batch + b) * W;
                if (d == depths - 1) {
                    size_t cs = ((size_t)l * batch + b) * capacity;
                    memcpy(k_top + (cs + p) * row, k_new + ss * row, sizeof(uint16_t) * n * row);
                    memcpy(v_top + (cs + p) * row, v_new + ss * row, sizeof(uint16_t) * n * row);
                } else {
                    size_t cs = (((size_t)d * layers + l) * batch + b) * capacity;
                    das_oracle_e4m3_from_bf16_n(k_new + ss * row, k_low + (cs + p) * row, n * row);
                    das_oracle_e4m3_from_bf16_n(v_new + ss * row, v_low + (cs + p) * row, n * row);
                }
            }
        prefix_len[b] = p + n;
    }
}
