/*
 * jb_oracle.c -- plain, slow CPU oracle for the seeded-perturbation hot path of
 * "Just One Byte (per gradient)" (arXiv 2306.10015).
 *
 * TEST INFRASTRUCTURE. Only the tests, the smoke check and the benchmark's CPU
 * baseline may load this library. The product (the CUDA path) shares no code,
 * header, table or constant with it and never calls it.
 *
 * Everything is computed in double precision, element by element, in the
 * order the paper states the method:
 *   - PerturbParameters(theta, eps, s): reseed, draw z ~ N(0,1) per parameter,
 *     theta_i += eps * z_i                      (Algorithm 1, subroutine)
 *   - the SPSA sample +eps, -2eps, +eps around two losses
 *                                               (Algorithm 1, inference loop)
 *   - apply every machine's projected gradients in machine-timestamp order
 *     with weight minus gradient times learning rate over the number of gradients
 *                                               (Algorithm 1; Section 2)
 *   - the one-byte signed-log projected gradient clipped to +-127
 *                                               (Section 3, Training Speed)
 *
 * Readings where the paper is silent (it names no generator, Appendix B says
 * only that PyTorch's CUDA generator is used and is not portable):
 *   - generator: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random
 *     numbers: as easy as 1, 2, 3", SC 2011), key = machine id (lo, hi word),
 *     counter = (block lo, block hi, step, sample id), block = element >> 2,
 *     element e uses word e & 3 of its block;
 *   - uniforms: u_a = ((x >> 9) + 0.5) * 2^-23 for the radius word and
 *     u_b = ((x >> 8) + 0.5) * 2^-24 for the angle word (both strictly inside
 *     (0, 1));
 *   - Box-Muller (Box & Muller 1958) on words (0,1) and (2,3):
 *     r = sqrt(-2 ln u_a), even element r cos(2 pi u_b), odd element
 *     r sin(2 pi u_b);
 *   - perturb result: one rounding of theta + eps z to the storage type;
 *   - update: one rounding of theta + sum_k c_k z_k, c_k = f32(-lr deq(q_k) /
 *     denom), seeds in ascending (machine id, step, sample id) order;
 *   - byte code: q = sign(g) min(127, round_half_away(S ln(1 + |g|))),
 *     deq(q) = sign(q) expm1(|q| / S), code -128 decodes as -127.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#include "jb_oracle.h"

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon et al. 2011): a 4-word counter, a 2-word key, ten    */
/* rounds. Each round multiplies words 0 and 2 by two odd constants into      */
/* 64-bit products and mixes the high halves with the other words and the     */
/* key; the key is bumped by two Weyl constants between rounds.               */
/* ------------------------------------------------------------------------ */
static const uint32_t PHILOX_M0 = 0xD2511F53u;
static const uint32_t PHILOX_M1 = 0xCD9E8D57u;
static const uint32_t PHILOX_W0 = 0x9E3779B9u; /* golden ratio */
static const uint32_t PHILOX_W1 = 0xBB67AE85u; /* sqrt(3) - 1 */

void jbo_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += PHILOX_W0;
            k1 += PHILOX_W1;
        }
        uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)x0;
        uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)x2;
        uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
        uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
        x0 = hi1 ^ x1 ^ k0;
        x1 = lo1;
        x2 = hi0 ^ x3 ^ k1;
        x3 = lo0;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* Seed s = (machine time id, iteration, sample index) of Algorithm 1 mapped to
 * the Philox key and counter of block b. */
void jbo_block_words(jbo_seed s, uint64_t block, uint32_t out[4]) {
    uint32_t ctr[4], key[2];
    ctr[0] = (uint32_t)block;
    ctr[1] = (uint32_t)(block >> 32);
    ctr[2] = s.step;
    ctr[3] = s.sample_id;
    key[0] = (uint32_t)s.machine_id;
    key[1] = (uint32_t)(s.machine_id >> 32);
    jbo_philox4x32_10(ctr, key, out);
}

void jbo_philox_blocks(jbo_seed s, uint64_t first_block, uint64_t n_blocks, uint32_t* out) {
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n_blocks; ++i)
        jbo_block_words(s, first_block + (uint64_t)i, out + 4 * i);
}

/* ------------------------------------------------------------------------ */
/* Uniforms and the Box-Muller transform.                                    */
/* ------------------------------------------------------------------------ */
double jbo_uniform_a(uint32_t x) { return ((double)(x >> 9) + 0.5) * 0x1p-23; }
double jbo_uniform_b(uint32_t x) { return ((double)(x >> 8) + 0.5) * 0x1p-24; }

/* (z_even, z_odd) = sqrt(-2 ln u_a) * (cos 2 pi u_b, sin 2 pi u_b). */
void jbo_box_muller(uint32_t xa, uint32_t xb, double out[2]) {
    const double two_pi = 6.283185307179586476925286766559;
    double r = sqrt(-2.0 * log(jbo_uniform_a(xa)));
    double angle = two_pi * jbo_uniform_b(xb);
    out[0] = r * cos(angle);
    out[1] = r * sin(angle);
}

/* z ~ N(0,1) drawn for global element index e under seed s. */
double jbo_gaussian(jbo_seed s, uint64_t e) {
    uint32_t w[4];
    double z[2];
    jbo_block_words(s, e >> 2, w);
    unsigned pair = (unsigned)((e >> 1) & 1u);
    jbo_box_muller(w[2 * pair], w[2 * pair + 1], z);
    return z[e & 1u];
}

void jbo_gaussian_range(jbo_seed s, uint64_t first, uint64_t n, double* out) {
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) out[i] = jbo_gaussian(s, first + (uint64_t)i);
}

void jbo_gaussian_at(jbo_seed s, const uint64_t* idx, uint64_t n, double* out) {
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) out[i] = jbo_gaussian(s, idx[i]);
}

void jbo_box_muller_pairs(const uint32_t* words, uint64_t n_pairs, double* out) {
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n_pairs; ++i)
        jbo_box_muller(words[2 * i], words[2 * i + 1], out + 2 * i);
}

/* ------------------------------------------------------------------------ */
/* Storage types: fp32 and bf16 (8 significant bits, fp32 exponent range),   */
/* rounding to nearest, ties to even, from a double.                          */
/* ------------------------------------------------------------------------ */
uint16_t jbo_round_bf16(double x) {
    if (isnan(x)) return 0x7FC0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (a == 0.0) return sign;
    int e;
    frexp(a, &e);                /* a = m 2^e, 0.5 <= m < 1 */
    int q = e - 8;               /* quantum 2^q keeps 8 significant bits */
    if (q < -133) q = -133;      /* subnormal quantum of the fp32 exponent range */
    double r = nearbyint(ldexp(a, -q)); /* ties to even in the default mode */
    double v = ldexp(r, q);
    if (v >= 0x1p128) return (uint16_t)(sign | 0x7F80);
    float f = (float)v;          /* exact: v has <= 8 significant bits */
    uint32_t bits;
    memcpy(&bits, &f, 4);
    return (uint16_t)(sign | ((bits >> 16) & 0x7FFF));
}

double jbo_bf16_to_double(uint16_t h) {
    uint32_t bits = (uint32_t)h << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
}

static double load_theta(const void* theta, int dtype, uint64_t i) {
    if (dtype == JBO_F32) return (double)((const float*)theta)[i];
    return jbo_bf16_to_double(((const uint16_t*)theta)[i]);
}

static void store_theta(void* theta, int dtype, uint64_t i, double v) {
    if (dtype == JBO_F32) ((float*)theta)[i] = (float)v; /* one rounding, nearest-even */
    else ((uint16_t*)theta)[i] = jbo_round_bf16(v);
}

/* PerturbParameters(theta, eps, s) over a tensor whose element i has global
 * index flat_offset + i (Algorithm 1, subroutine). In place. */
void jbo_perturb(void* theta, int dtype, uint64_t n, uint64_t flat_offset, jbo_seed s, double eps) {
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) {
        double t = load_theta(theta, dtype, (uint64_t)i);
        double z = jbo_gaussian(s, flat_offset + (uint64_t)i);
        store_theta(theta, dtype, (uint64_t)i, t + eps * z);
    }
}

/* Same, for sampled global indices: out[j] = perturbed value of element idx[j]
 * whose value before the call was in[j]. */
void jbo_perturb_at(const void* in, void* out, int dtype, const uint64_t* idx, uint64_t n,
                    jbo_seed s, double eps) {
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < (int64_t)n; ++j) {
        double t = load_theta(in, dtype, (uint64_t)j);
        store_theta(out, dtype, (uint64_t)j, t + eps * jbo_gaussian(s, idx[j]));
    }
}

/* ------------------------------------------------------------------------ */
/* One-byte projected gradient (Section 3, Training Speed).                   */
/* ------------------------------------------------------------------------ */
int8_t jbo_quantize(double g, double qscale) {
    if (isnan(g)) return 0;
    double mag = isinf(g) ? 127.0 : round(qscale * log1p(fabs(g)));
    if (mag > 127.0) mag = 127.0;
    int q = (int)mag;
    return (int8_t)(g < 0 ? -q : q);
}

double jbo_dequantize(int8_t q, double qscale) {
    int m = q < 0 ? -(int)q : (int)q;
    if (m > 127) m = 127;
    double v = expm1((double)m / qscale);
    return q < 0 ? -v : v;
}

/* Weight of one projected gradient in the step update: -grad * eta / numel
 * (Algorithm 1), with grad the dequantized byte; rounded once to fp32. */
float jbo_coefficient(int8_t q, double lr, double denom, double qscale) {
    return (float)(-lr * jbo_dequantize(q, qscale) / denom);
}

/* ------------------------------------------------------------------------ */
/* The step update: every machine's projected gradients, taken in the order  */
/* of the machines' start times (Section 2; Algorithm 1).                     */
/* ------------------------------------------------------------------------ */
static int seed_cmp(const jbo_seed* a, const jbo_seed* b) {
    if (a->machine_id != b->machine_id) return a->machine_id < b->machine_id ? -1 : 1;
    if (a->step != b->step) return a->step < b->step ? -1 : 1;
    if (a->sample_id != b->sample_id) return a->sample_id < b->sample_id ? -1 : 1;
    return 0;
}

/* perm = indices of seeds in ascending (machine id, step, sample id) order.
 * Returns -1 if two seeds are equal, else 0. Insertion sort: K is small. */
int jbo_canonical_order(const jbo_seed* seeds, int K, int* perm) {
    for (int i = 0; i < K; ++i) perm[i] = i;
    for (int i = 1; i < K; ++i) {
        int p = perm[i], j = i - 1;
        while (j >= 0 && seed_cmp(&seeds[perm[j]], &seeds[p]) > 0) {
            perm[j + 1] = perm[j];
            --j;
        }
        perm[j + 1] = p;
    }
    for (int i = 1; i < K; ++i)
        if (seed_cmp(&seeds[perm[i - 1]], &seeds[perm[i]]) == 0) return -1;
    return 0;
}

static int prepare_update(const jbo_seed* seeds, const int8_t* q, int K, double lr, double denom,
                          double qscale, jbo_seed* s_sorted, double* c_sorted) {
    int* perm = (int*)malloc(sizeof(int) * (size_t)(K > 0 ? K : 1));
    if (!perm) return -2;
    int rc = jbo_canonical_order(seeds, K, perm);
    for (int i = 0; rc == 0 && i < K; ++i) {
        s_sorted[i] = seeds[perm[i]];
        c_sorted[i] = (double)jbo_coefficient(q[perm[i]], lr, denom, qscale);
    }
    free(perm);
    return rc;
}

/* theta_e <- round(theta_e + sum_k c_k z_k(e)); in place over one tensor. */
int jbo_update(void* theta, int dtype, uint64_t n, uint64_t flat_offset, const jbo_seed* seeds,
               const int8_t* q, int K, double lr, double denom, double qscale) {
    jbo_seed* ss = (jbo_seed*)malloc(sizeof(jbo_seed) * (size_t)(K > 0 ? K : 1));
    double* cc = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
    if (!ss || !cc) { free(ss); free(cc); return -2; }
    int rc = prepare_update(seeds, q, K, lr, denom, qscale, ss, cc);
    if (rc == 0) {
        #pragma omp parallel for schedule(static)
        for (int64_t i = 0; i < (int64_t)n; ++i) {
            double acc = 0.0;
            for (int k = 0; k < K; ++k) acc += cc[k] * jbo_gaussian(ss[k], flat_offset + (uint64_t)i);
            store_theta(theta, dtype, (uint64_t)i, load_theta(theta, dtype, (uint64_t)i) + acc);
        }
    }
    free(ss); free(cc);
    return rc;
}

/* Same, for sampled global indices (in[j] is the value of element idx[j]). */
int jbo_update_at(const void* in, void* out, int dtype, const uint64_t* idx, uint64_t n,
                  const jbo_seed* seeds, const int8_t* q, int K, double lr, double denom,
                  double qscale) {
    jbo_seed* ss = (jbo_seed*)malloc(sizeof(jbo_seed) * (size_t)(K > 0 ? K : 1));
    double* cc = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
    if (!ss || !cc) { free(ss); free(cc); return -2; }
    int rc = prepare_update(seeds, q, K, lr, denom, qscale, ss, cc);
    if (rc == 0) {
        #pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < (int64_t)n; ++j) {
            double acc = 0.0;
            for (int k = 0; k < K; ++k) acc += cc[k] * jbo_gaussian(ss[k], idx[j]);
            store_theta(out, dtype, (uint64_t)j, load_theta(in, dtype, (uint64_t)j) + acc);
        }
    }
    free(ss); free(cc);
    return rc;
}

/* Sum_k c_k z_k(e) in double for sampled indices (no rounding to storage). */
int jbo_update_delta_at(const uint64_t* idx, uint64_t n, const jbo_seed* seeds, const int8_t* q,
                        int K, double lr, double denom, double qscale, double* out) {
    jbo_seed* ss = (jbo_seed*)malloc(sizeof(jbo_seed) * (size_t)(K > 0 ? K : 1));
    double* cc = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
    if (!ss || !cc) { free(ss); free(cc); return -2; }
    int rc = prepare_update(seeds, q, K, lr, denom, qscale, ss, cc);
    if (rc == 0) {
        #pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < (int64_t)n; ++j) {
            double acc = 0.0;
            for (int k = 0; k < K; ++k) acc += cc[k] * jbo_gaussian(ss[k], idx[j]);
            out[j] = acc;
        }
    }
    free(ss); free(cc);
    return rc;
}

/* The same sum together with sum_k |c_k z_k(e)| (the size of the operands,
 * which the parity tolerances scale with), from one evaluation of each z. */
int jbo_update_delta_abs_at(const uint64_t* idx, uint64_t n, const jbo_seed* seeds,
                            const int8_t* q, int K, double lr, double denom, double qscale,
                            double* out, double* out_abs) {
    jbo_seed* ss = (jbo_seed*)malloc(sizeof(jbo_seed) * (size_t)(K > 0 ? K : 1));
    double* cc = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
    if (!ss || !cc) { free(ss); free(cc); return -2; }
    int rc = prepare_update(seeds, q, K, lr, denom, qscale, ss, cc);
    if (rc == 0) {
        #pragma omp parallel for schedule(static)
        for (int64_t j = 0; j < (int64_t)n; ++j) {
            double acc = 0.0, mag = 0.0;
            for (int k = 0; k < K; ++k) {
                const double t = cc[k] * jbo_gaussian(ss[k], idx[j]);
                acc += t;
                mag += fabs(t);
            }
            out[j] = acc;
            out_abs[j] = mag;
        }
    }
    free(ss); free(cc);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* 4-bit weights (Section 3, Training Speed: weights are dequantized before   */
/* the noise is added and quantized again). Reading (the paper fixes no       */
/* format; it cites QLoRA's NormalFloat): 16 levels built from quantiles of   */
/* N(0,1), 8 at probabilities delta + (1/2 - delta) j/7 (j = 0..7, the last   */
/* is the median 0) and 8 more at 1/2 + (1/2 - delta) j/8 (j = 1..8), divided */
/* by the largest so they span [-1, 1]; delta = 1/32. Levels are stored as    */
/* fp32. Blocks of 64 elements share one fp32 scale, the largest |w| of the   */
/* block; code = number of midpoints between adjacent levels lying strictly   */
/* below w / scale (the nearest level, ties to the lower). Element 2i sits in */
/* the low nibble of byte i.                                                  */
/* ------------------------------------------------------------------------ */
static double std_normal_quantile(double p) {
    /* bisection on Phi(x) = erfc(-x / sqrt 2) / 2, to double precision */
    double lo = -40.0, hi = 40.0;
    for (int it = 0; it < 200; ++it) {
        double mid = 0.5 * (lo + hi);
        double phi = 0.5 * erfc(-mid / sqrt(2.0));
        if (phi < p) lo = mid; else hi = mid;
    }
    return 0.5 * (lo + hi);
}

void jbo_q4_levels(float out[16]) {
    const double delta = 1.0 / 32.0;
    double v[16];
    for (int j = 0; j < 8; ++j) v[j] = std_normal_quantile(delta + (0.5 - delta) * j / 7.0);
    v[7] = 0.0;
    for (int j = 1; j <= 8; ++j) v[7 + j] = std_normal_quantile(0.5 + (0.5 - delta) * j / 8.0);
    double top = v[15];
    for (int j = 0; j < 16; ++j) out[j] = (float)(v[j] / top);
    out[7] = 0.0f;
    out[15] = 1.0f;
}

static unsigned q4_code(double x, const float lev[16]) {
    unsigned c = 0;
    for (int j = 0; j < 15; ++j)
        if (x > 0.5 * ((double)lev[j] + (double)lev[j + 1])) c = (unsigned)j + 1;
    return c;
}

/* Quantize n values (a tensor) into codes (n + 1) / 2 bytes and scales per 64. */
void jbo_q4_quantize(const double* w, uint64_t n, uint8_t* codes, float* scale) {
    float lev[16];
    jbo_q4_levels(lev);
    for (uint64_t b = 0; b * 64 < n; ++b) {
        uint64_t end = (b + 1) * 64 < n ? (b + 1) * 64 : n;
        double m = 0.0;
        for (uint64_t i = b * 64; i < end; ++i) if (fabs(w[i]) > m) m = fabs(w[i]);
        scale[b] = (float)m;
        for (uint64_t i = b * 64; i < end; ++i) {
            unsigned c = q4_code(m > 0.0 ? w[i] / (double)scale[b] : 0.0, lev);
            if (i % 2 == 0) codes[i / 2] = (uint8_t)((codes[i / 2] & 0xF0u) | c);
            else codes[i / 2] = (uint8_t)((codes[i / 2] & 0x0Fu) | (c << 4));
        }
    }
}

void jbo_q4_dequantize(const uint8_t* codes, const float* scale, uint64_t n, double* w) {
    float lev[16];
    jbo_q4_levels(lev);
    for (uint64_t i = 0; i < n; ++i) {
        unsigned c = (i % 2 == 0) ? (codes[i / 2] & 0x0Fu) : (codes[i / 2] >> 4);
        w[i] = (double)lev[c] * (double)scale[i / 64];
    }
}

/* PerturbParameters on 4-bit weights: dequantize, add eps z, quantize again.
 * Also returns the perturbed values before quantization in w_out (may be NULL). */
int jbo_q4_perturb(uint8_t* codes, float* scale, uint64_t n, uint64_t flat_offset, jbo_seed s,
                   double eps, double* w_out) {
    double* w = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    if (!w) return -2;
    jbo_q4_dequantize(codes, scale, n, w);
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) w[i] += eps * jbo_gaussian(s, flat_offset + (uint64_t)i);
    jbo_q4_quantize(w, n, codes, scale);
    if (w_out) memcpy(w_out, w, sizeof(double) * (size_t)n);
    free(w);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Model checksum for ChecksumMatch (Algorithm 1: "check if hashed theta      */
/* matches peer's"). The paper fixes no hash. Reading: the global element     */
/* index space is cut into windows of 16 bytes of storage (8 bf16 or 4 fp32   */
/* elements; window v = elements [vE, vE + E)). Each window that overlaps a   */
/* segment contributes, per segment, the first four Philox4x32 rounds of its  */
/* four storage words (elements outside the segment read as 0) under the key */
/* (lo v, hi v) xor (0x6A09E667, 0xF3BCC908); the checksum is the sum mod     */
/* 2^64 of (x1:x0) + (x3:x2) over all contributions. Four rounds carry every */
/* input bit into every output word; the sum does not depend on the order in  */
/* which windows are evaluated.                                               */
/* ------------------------------------------------------------------------ */
static void philox_rounds(uint32_t w[4], uint32_t k0, uint32_t k1, int rounds) {
    for (int r = 0; r < rounds; ++r) {
        if (r > 0) {
            k0 += PHILOX_W0;
            k1 += PHILOX_W1;
        }
        uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)w[0];
        uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)w[2];
        uint32_t y0 = (uint32_t)(p1 >> 32) ^ w[1] ^ k0;
        uint32_t y2 = (uint32_t)(p0 >> 32) ^ w[3] ^ k1;
        w[1] = (uint32_t)p1;
        w[3] = (uint32_t)p0;
        w[0] = y0;
        w[2] = y2;
    }
}

uint64_t jbo_window_hash(uint64_t window, const uint32_t words[4]) {
    uint32_t w[4] = {words[0], words[1], words[2], words[3]};
    philox_rounds(w, (uint32_t)window ^ 0x6A09E667u, (uint32_t)(window >> 32) ^ 0xF3BCC908u, 4);
    return ((uint64_t)w[1] << 32 | w[0]) + ((uint64_t)w[3] << 32 | w[2]);
}

/* Contribution of one segment (values at global indices fo .. fo + n - 1). */
uint64_t jbo_checksum_segment(const void* theta, int dtype, uint64_t n, uint64_t fo) {
    const uint64_t E = dtype == JBO_F32 ? 4 : 8;
    uint64_t sum = 0;
    if (n == 0) return 0;
    for (uint64_t v = fo / E; v <= (fo + n - 1) / E; ++v) {
        uint32_t words[4] = {0, 0, 0, 0};
        for (uint64_t t = 0; t < E; ++t) {
            uint64_t e = v * E + t;
            if (e < fo || e >= fo + n) continue;
            uint64_t i = e - fo;
            if (dtype == JBO_F32) {
                uint32_t b;
                memcpy(&b, (const float*)theta + i, 4);
                words[t] = b;
            } else {
                uint32_t b = ((const uint16_t*)theta)[i];
                words[t / 2] |= b << (16 * (t % 2));
            }
        }
        sum += jbo_window_hash(v, words);
    }
    return sum;
}

/* ------------------------------------------------------------------------ */
/* Threads                                                                    */
/* ------------------------------------------------------------------------ */
void jbo_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int jbo_get_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
