/*
 * synth_core.h -- seeded, counter-based synthetic inputs for the DAS hot path.
 *
 * This is the one module that both the CUDA path (device fill, benchmarks)
 * and the CPU oracle's tests (host generation) use.  It holds no attention,
 * softmax, argmax or cache-commit arithmetic: it only turns (seed, tensor,
 * coordinates) into numbers.  The same source compiles for the host (C,
 * -ffp-contract=off) and the device (CUDA, --fmad=false), and uses only
 * correctly rounded IEEE operations (+ - * / sqrt) and integer operations, so
 * both sides produce bit-identical values.
 *
 * Definitions
 *   mix(z)       SplitMix64 output function (Steele, Lea & Flood, "Fast
 *                splittable pseudorandom number generators", OOPSLA 2014),
 *                with the multipliers of the public-domain splitmix64.c.
 *   stream       a SplitMix64 stream with initial state s yields
 *                mix(s + n*GAMMA) as its n-th output (n >= 1).
 *   key(seed,t)  the state of the stream of tensor t: mix(mix(seed) + t*GAMMA).
 *   normal(k,c)  Box-Muller (1958) on the stream's outputs 2c+1 and 2c+2:
 *                u1 = (top 53 bits + 1) * 2^-53 in (0,1],
 *                u2 = (top 53 bits) * 2^-53 in [0,1),
 *                sqrt(-2 ln u1) * cos(2 pi u2).
 *                ln uses the atanh series ln m = 2 sum s^(2k+1)/(2k+1),
 *                s = (m-1)/(m+1), after m in [sqrt(1/2), sqrt(2));
 *                cos uses exact quarter/eighth-turn symmetries and the Taylor
 *                series of cos and sin on [0, pi/4].  Accuracy ~1e-16 rel.
 *   maturation   for stored depth d of R (1..R): X_d = X_R + c(d) * N_d with
 *                c_K(d) = (1 - d/R)^3 for keys, c_V(d) = (1 - d/R)^1.5 for
 *                values; X_R and N_d are independent N(0,1) draws
 *                (component 0 is X_R, component d is N_d).
 *   bf16         one round-to-nearest-even of the double to bfloat16.
 */
#ifndef DAS_SYNTH_CORE_H
#define DAS_SYNTH_CORE_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYNTH_FN static __host__ __device__ __forceinline__
#define SYNTH_SQRT(x) sqrt(x)
#else
#include <math.h>
#define SYNTH_FN static inline
#define SYNTH_SQRT(x) sqrt(x)
#endif

#define SYNTH_GAMMA 0x9E3779B97F4A7C15ULL

/* tensor ids (each has its own stream) */
enum {
    SYNTH_T_KCACHE = 1,
    SYNTH_T_VCACHE = 2,
    SYNTH_T_Q = 3,
    SYNTH_T_KBLK = 4,
    SYNTH_T_VBLK = 5,
    SYNTH_T_KNEW = 6,
    SYNTH_T_VNEW = 7,
    SYNTH_T_LOGITS = 8,
    SYNTH_T_DRAFT = 9,
    SYNTH_T_ACCEPT = 10,
    SYNTH_T_PREFIX = 11,
    SYNTH_T_BLOCK = 12,
    SYNTH_T_FILL = 13,
    SYNTH_T_KLOW = 14,
    SYNTH_T_VLOW = 15
};

SYNTH_FN uint64_t synth_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

SYNTH_FN uint64_t synth_key(uint64_t seed, uint64_t tensor) {
    return synth_mix(synth_mix(seed) + tensor * SYNTH_GAMMA);
}

/* n-th output (n >= 1) of the stream with state `key` */
SYNTH_FN uint64_t synth_out(uint64_t key, uint64_t n) { return synth_mix(key + n * SYNTH_GAMMA); }

/* Coordinates of a cache-shaped element packed into one counter:
 * comp 6 bits | layer 6 | batch 8 | token 21 | head 8 | dim 9  (58 bits). */
SYNTH_FN uint64_t synth_ctr(uint32_t comp, uint32_t layer, uint32_t b, uint32_t tok,
                            uint32_t head, uint32_t dim) {
    return ((uint64_t)comp << 52) | ((uint64_t)layer << 46) | ((uint64_t)b << 38) |
           ((uint64_t)tok << 17) | ((uint64_t)head << 9) | (uint64_t)dim;
}

/* 2^k for integer k in [-1022, 1023], built from bits */
SYNTH_FN double synth_pow2(int k) {
    union { uint64_t u; double d; } v;
    v.u = (uint64_t)(k + 1023) << 52;
    return v.d;
}

/* natural log of x in (0, 1], x a normal double */
SYNTH_FN double synth_ln(double x) {
    union { double d; uint64_t u; } v;
    v.d = x;
    int e = (int)((v.u >> 52) & 0x7FF) - 1023;
    v.u = (v.u & 0x000FFFFFFFFFFFFFULL) | 0x3FF0000000000000ULL; /* m in [1,2) */
    double m = v.d;
    /* 1.4142135623730951 is the double nearest sqrt(2) */
    if (m > 1.4142135623730951) {
        m = m * 0.5;
        e = e + 1;
    }
    double s = (m - 1.0) / (m + 1.0);
    double s2 = s * s;
    double poly = 1.0 / 25.0;
    for (int k = 23; k >= 1; k -= 2) poly = poly * s2 + 1.0 / (double)k;
    double ln_m = 2.0 * s * poly;
    /* 0.6931471805599453 is the double nearest ln 2 */
    return (double)e * 0.6931471805599453 + ln_m;
}

/* cos(x) and sin(x) for x in [0, pi/4] by their Taylor series */
SYNTH_FN double synth_cos_series(double x) {
    double x2 = x * x, term = 1.0, sum = 1.0;
    for (int k = 1; k <= 11; ++k) {
        term = term * (-x2) / (double)((2 * k - 1) * (2 * k));
        sum = sum + term;
    }
    return sum;
}
SYNTH_FN double synth_sin_series(double x) {
    double x2 = x * x, term = x, sum = x;
    for (int k = 1; k <= 11; ++k) {
        term = term * (-x2) / (double)((2 * k) * (2 * k + 1));
        sum = sum + term;
    }
    return sum;
}

/* cos(2 pi u) for u in [0, 1); every reduction step below is exact */
SYNTH_FN double synth_cos_turn(double u) {
    double sign = 1.0;
    if (u > 0.5) u = 1.0 - u;       /* cos(2pi u) = cos(2pi (1-u)) */
    if (u > 0.25) {                 /* cos(2pi u) = -cos(2pi (1/2-u)) */
        u = 0.5 - u;
        sign = -1.0;
    }
    /* 6.283185307179586 is the double nearest 2 pi */
    if (u > 0.125) return sign * synth_sin_series(6.283185307179586 * (0.25 - u));
    return sign * synth_cos_series(6.283185307179586 * u);
}

/* standard normal at counter c of the stream with state key */
SYNTH_FN double synth_normal(uint64_t key, uint64_t c) {
    uint64_t h1 = synth_out(key, 2 * c + 1);
    uint64_t h2 = synth_out(key, 2 * c + 2);
    double u1 = (double)((h1 >> 11) + 1) * synth_pow2(-53);
    double u2 = (double)(h2 >> 11) * synth_pow2(-53);
    return SYNTH_SQRT(-2.0 * synth_ln(u1)) * synth_cos_turn(u2);
}

/* depth-maturation coefficient: is_value ? (1-d/R)^1.5 : (1-d/R)^3 */
SYNTH_FN double synth_maturity_coef(int is_value, int d, int R) {
    double t = (double)(R - d) / (double)R;
    return is_value ? t * SYNTH_SQRT(t) : t * t * t;
}

/* one element at stored depth d (1..R) under the maturation law */
SYNTH_FN double synth_matured(uint64_t key, int is_value, int d, int R, uint32_t layer,
                              uint32_t b, uint32_t tok, uint32_t head, uint32_t dim) {
    double base = synth_normal(key, synth_ctr(0, layer, b, tok, head, dim));
    if (d >= R) return base;
    double noise = synth_normal(key, synth_ctr((uint32_t)d, layer, b, tok, head, dim));
    return base + synth_maturity_coef(is_value, d, R) * noise;
}

/* double -> bfloat16 bits, one round-to-nearest-even */
SYNTH_FN uint16_t synth_bf16(double x) {
    union { double d; uint64_t u; } v;
    v.d = x;
    uint16_t sign = (uint16_t)((v.u >> 63) << 15);
    int ex = (int)((v.u >> 52) & 0x7FF);
    uint64_t mant = v.u & 0x000FFFFFFFFFFFFFULL;
    if (ex == 0x7FF) return (uint16_t)(sign | (mant ? 0x7FC0 : 0x7F80));
    if (ex == 0) return sign; /* |x| < 2^-1022 rounds to zero in bf16 */
    int e = ex - 1023;
    uint64_t m = mant | (1ULL << 52); /* 53-bit significand */
    int shift;                        /* bits dropped from m */
    if (e >= -126) {
        shift = 45; /* keep 1 + 7 bits */
    } else {
        shift = -81 - e; /* subnormal: m * 2^(e-52) / 2^-133 */
        if (shift > 60) return sign;
    }
    uint64_t q = m >> shift;
    uint64_t rem = m & ((1ULL << shift) - 1);
    uint64_t half = 1ULL << (shift - 1);
    if (rem > half || (rem == half && (q & 1))) q++;
    if (e >= -126) {
        if (q == 256) {
            q = 128;
            e++;
        }
        if (e > 127) return (uint16_t)(sign | 0x7F80);
        return (uint16_t)(sign | ((uint16_t)(e + 127) << 7) | (uint16_t)(q & 0x7F));
    }
    return (uint16_t)(sign | (uint16_t)q); /* q == 128 is the smallest normal */
}

#endif /* DAS_SYNTH_CORE_H */
