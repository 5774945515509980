/*
 * jb_oracle.h -- declarations of the CPU oracle (test infrastructure only).
 * Double-precision restatement of the seeded perturbation, the step update and
 * the one-byte projected gradient of "Just One Byte (per gradient)"
 * (arXiv 2306.10015, Algorithm 1 and Section 3). See jb_oracle.c.
 */
#ifndef JB_ORACLE_H
#define JB_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { JBO_F32 = 0, JBO_BF16 = 1 };

/* Seed of Algorithm 1: (machine start-time id, iteration, sample index). */
typedef struct {
    uint64_t machine_id;
    uint32_t step;
    uint32_t sample_id;
} jbo_seed;

void jbo_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
void jbo_block_words(jbo_seed s, uint64_t block, uint32_t out[4]);
void jbo_philox_blocks(jbo_seed s, uint64_t first_block, uint64_t n_blocks, uint32_t* out);

double jbo_uniform_a(uint32_t x);
double jbo_uniform_b(uint32_t x);
void jbo_box_muller(uint32_t xa, uint32_t xb, double out[2]);
void jbo_box_muller_pairs(const uint32_t* words, uint64_t n_pairs, double* out);
double jbo_gaussian(jbo_seed s, uint64_t e);
void jbo_gaussian_range(jbo_seed s, uint64_t first, uint64_t n, double* out);
void jbo_gaussian_at(jbo_seed s, const uint64_t* idx, uint64_t n, double* out);

uint16_t jbo_round_bf16(double x);
double jbo_bf16_to_double(uint16_t h);

void jbo_perturb(void* theta, int dtype, uint64_t n, uint64_t flat_offset, jbo_seed s, double eps);
void jbo_perturb_at(const void* in, void* out, int dtype, const uint64_t* idx, uint64_t n,
                    jbo_seed s, double eps);

int8_t jbo_quantize(double g, double qscale);
double jbo_dequantize(int8_t q, double qscale);
float jbo_coefficient(int8_t q, double lr, double denom, double qscale);

int jbo_canonical_order(const jbo_seed* seeds, int K, int* perm);
int jbo_update(void* theta, int dtype, uint64_t n, uint64_t flat_offset, const jbo_seed* seeds,
               const int8_t* q, int K, double lr, double denom, double qscale);
int jbo_update_at(const void* in, void* out, int dtype, const uint64_t* idx, uint64_t n,
                  const jbo_seed* seeds, const int8_t* q, int K, double lr, double denom,
                  double qscale);
int jbo_update_delta_at(const uint64_t* idx, uint64_t n, const jbo_seed* seeds, const int8_t* q,
                        int K, double lr, double denom, double qscale, double* out);
int jbo_update_delta_abs_at(const uint64_t* idx, uint64_t n, const jbo_seed* seeds,
                            const int8_t* q, int K, double lr, double denom, double qscale,
                            double* out, double* out_abs);

void jbo_q4_levels(float out[16]);
void jbo_q4_quantize(const double* w, uint64_t n, uint8_t* codes, float* scale);
void jbo_q4_dequantize(const uint8_t* codes, const float* scale, uint64_t n, double* w);
int jbo_q4_perturb(uint8_t* codes, float* scale, uint64_t n, uint64_t flat_offset, jbo_seed s,
                   double eps, double* w_out);

uint64_t jbo_window_hash(uint64_t window, const uint32_t words[4]);
uint64_t jbo_checksum_segment(const void* theta, int dtype, uint64_t n, uint64_t fo);

void jbo_set_threads(int n);
int jbo_get_threads(void);

#ifdef __cplusplus
}
#endif
#endif
