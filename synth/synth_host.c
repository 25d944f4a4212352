/*
 * synth_host.c -- host side of the seeded input generator (see synth_core.h).
 * Built with -ffp-contract=off so that it matches the device side bit for bit.
 * Every function returns 0 on success and 1 on coordinates the counter layout
 * cannot hold.
 */
#include <pthread.h>
#include <stdlib.h>

#include "synth_core.h"

static int coords_ok(int comp, int layer, int b, int tok_hi, int head_hi, int D) {
    return comp >= 0 && comp < 64 && layer >= 0 && layer < 64 && b >= 0 && b < 256 &&
           tok_hi <= (1 << 21) && head_hi <= 256 && D > 0 && D <= 512;
}

typedef struct {
    uint64_t key;
    int is_value, depth, R, layer, b, t0, t1, h0, h1, D;
    double divisor; /* normal-only mode when depth == 0 */
    uint16_t *out;
    int next;
    pthread_mutex_t mu;
} block_job;

static void *block_worker(void *arg) {
    block_job *J = (block_job *)arg;
    int nh = J->h1 - J->h0;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        int t = J->t0 + J->next++;
        pthread_mutex_unlock(&J->mu);
        if (t >= J->t1) break;
        uint16_t *row = J->out + (size_t)(t - J->t0) * nh * J->D;
        for (int h = J->h0; h < J->h1; ++h)
            for (int e = 0; e < J->D; ++e) {
                double x;
                if (J->depth > 0)
                    x = synth_matured(J->key, J->is_value, J->depth, J->R, (uint32_t)J->layer,
                                      (uint32_t)J->b, (uint32_t)t, (uint32_t)h, (uint32_t)e);
                else
                    x = synth_normal(J->key, synth_ctr(0, (uint32_t)J->layer, (uint32_t)J->b,
                                                       (uint32_t)t, (uint32_t)h, (uint32_t)e)) /
                        J->divisor;
                row[(size_t)(h - J->h0) * J->D + e] = synth_bf16(x);
            }
    }
    return NULL;
}

static int run_block(block_job *J, int nthreads) {
    J->next = 0;
    pthread_mutex_init(&J->mu, NULL);
    if (nthreads < 1) nthreads = 1;
    pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
    int started = 0;
    for (int i = 1; i < nthreads; ++i)
        if (pthread_create(&th[started], NULL, block_worker, J) == 0) ++started;
    block_worker(J);
    for (int i = 0; i < started; ++i) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&J->mu);
    return 0;
}

/*
 * Elements of a matured tensor (cache K/V, block K/V, staged K/V) at stored
 * depth `depth` (1..R), core layer, sequence b, tokens [t0,t1), heads [h0,h1),
 * all D dims.  out: bf16 bits [t1-t0][h1-h0][D].
 */
int synth_matured_block(uint64_t seed, int tensor, int is_value, int depth, int R, int layer,
                        int b, int t0, int t1, int h0, int h1, int D, uint16_t *out,
                        int nthreads) {
    if (depth < 1 || depth > R || R > 63 || t0 < 0 || t1 < t0 || h0 < 0 || h1 < h0 ||
        !coords_ok(depth, layer, b, t1, h1, D))
        return 1;
    block_job J;
    J.key = synth_key(seed, (uint64_t)tensor);
    J.is_value = is_value; J.depth = depth; J.R = R; J.layer = layer; J.b = b;
    J.t0 = t0; J.t1 = t1; J.h0 = h0; J.h1 = h1; J.D = D; J.divisor = 1.0; J.out = out;
    return run_block(&J, nthreads);
}

/* N(0,1)/divisor elements (queries use divisor sqrt(D)); layout as above. */
int synth_normal_block(uint64_t seed, int tensor, int layer, int b, int t0, int t1, int h0,
                       int h1, int D, double divisor, uint16_t *out, int nthreads) {
    if (t0 < 0 || t1 < t0 || h0 < 0 || h1 < h0 || !coords_ok(0, layer, b, t1, h1, D)) return 1;
    block_job J;
    J.key = synth_key(seed, (uint64_t)tensor);
    J.is_value = 0; J.depth = 0; J.R = 1; J.layer = layer; J.b = b;
    J.t0 = t0; J.t1 = t1; J.h0 = h0; J.h1 = h1; J.D = D; J.divisor = divisor; J.out = out;
    return run_block(&J, nthreads);
}

/* integer in [lo, hi] drawn from output idx+1 of tensor stream `tensor` */
int64_t synth_uniform_int(uint64_t seed, int tensor, uint64_t idx, int64_t lo, int64_t hi) {
    uint64_t span = (uint64_t)(hi - lo) + 1;
    return lo + (int64_t)(synth_out(synth_key(seed, (uint64_t)tensor), idx + 1) % span);
}

/*
 * Verifier logits and draft ids with a planted acceptance length.
 *   accept_star[b]  uniform in [0, W]
 *   draft[b][i]     uniform in [0, vocab)
 *   logits[b][i][v] = binary32(2 * N(0,1))   (variance 4)
 * then, for i < accept_star[b], logits[b][i][draft[b][i]] = +30 (so that the
 * draft id is the row's unique largest entry), and for i == accept_star[b] < W,
 * logits[b][i][draft[b][i]] = -30 (so that it is not).  A 2*N(0,1) draw
 * reaches |30| with probability below 1e-50.
 */
int synth_accept_inputs(uint64_t seed, int B, int W, int vocab, int32_t *accept_star,
                        int32_t *draft, float *logits) {
    if (B < 0 || W < 1 || vocab < 2) return 1;
    uint64_t kl = synth_key(seed, SYNTH_T_LOGITS);
    uint64_t kd = synth_key(seed, SYNTH_T_DRAFT);
    uint64_t ka = synth_key(seed, SYNTH_T_ACCEPT);
    for (int b = 0; b < B; ++b) {
        accept_star[b] = (int32_t)(synth_out(ka, (uint64_t)b + 1) % (uint64_t)(W + 1));
        for (int i = 0; i < W; ++i) {
            draft[b * W + i] =
                (int32_t)(synth_out(kd, (uint64_t)(b * W + i) + 1) % (uint64_t)vocab);
            float *row = logits + ((size_t)b * W + i) * vocab;
            for (int v = 0; v < vocab; ++v) {
                uint64_t c = ((uint64_t)b << 40) | ((uint64_t)i << 24) | (uint64_t)v;
                row[v] = (float)(2.0 * synth_normal(kl, c));
            }
            if (i < accept_star[b]) row[draft[b * W + i]] = 30.0f;
            else if (i == accept_star[b]) row[draft[b * W + i]] = -30.0f;
        }
    }
    return 0;
}

/* Element-wise access to the generator's primitives, for its own tests. */
void synth_bf16_array(const double *x, size_t n, uint16_t *out) {
    for (size_t i = 0; i < n; ++i) out[i] = synth_bf16(x[i]);
}
void synth_ln_array(const double *x, size_t n, double *out) {
    for (size_t i = 0; i < n; ++i) out[i] = synth_ln(x[i]);
}
void synth_cos_turn_array(const double *u, size_t n, double *out) {
    for (size_t i = 0; i < n; ++i) out[i] = synth_cos_turn(u[i]);
}
void synth_normal_array(uint64_t seed, int tensor, uint64_t c0, size_t n, double *out) {
    uint64_t key = synth_key(seed, (uint64_t)tensor);
    for (size_t i = 0; i < n; ++i) out[i] = synth_normal(key, c0 + i);
}

/*
 * 8-bit float codes for e4m3 cache contents, drawn (not rounded from
 * anything): out[i] = sign | exponent field | mantissa from output c0 + i + 1
 * of tensor stream `tensor`, with the exponent field in 4..9 (magnitudes
 * 2^-3 .. 1.875 * 2^2), so no code is NaN.
 */
void synth_e4m3_codes(uint64_t seed, int tensor, uint64_t c0, size_t n, uint8_t *out) {
    const uint64_t key = synth_key(seed, (uint64_t)tensor);
    for (size_t i = 0; i < n; ++i) {
        const uint64_t r = synth_out(key, c0 + i + 1);
        out[i] = (uint8_t)(((r >> 63) << 7) | ((4 + (r >> 40) % 6) << 3) | (r & 7));
    }
}
