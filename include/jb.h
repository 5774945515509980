/*
 * jb.h -- C ABI of the GB300 (sm_103a) seeded-perturbation library "libjb".
 *
 * The library implements the data-parallel hot path of the decentralized
 * shared-randomness SPSA of "Just One Byte (per gradient)" (arXiv 2306.10015):
 * regenerate a seeded Gaussian perturbation z over every model parameter, in
 * registers, and apply it in place.
 *
 *   jb_perturb        PerturbParameters(theta, eps, s): theta_i += eps z_i
 *                     (Algorithm 1, subroutine); called with +eps, -2 eps,
 *                     +eps around the two loss evaluations of one SPSA sample
 *                     (Algorithm 1, inference loop).
 *   jb_apply_updates  the step update: every machine's (seed, one-byte
 *                     projected gradient) pair applied with weight
 *                     minus the gradient times the learning rate over the
 *                     number of collected gradients, in machine-timestamp
 *                     order (Section 2, on applying the collected scalar projected
 *                     gradients; Algorithm 1), fused into one read and one
 *                     write of theta.
 *   jb_quantize_grad  the one-byte projected gradient: the logarithm of its
 *   jb_dequantize_grad magnitude with its sign, limited to +-127 (Section 3,
 *                     Training Speed).
 *
 * ---------------------------------------------------------------------------
 * Random stream. The paper names no generator (Appendix B notes that PyTorch's
 * CUDA generator is not reproducible across GPU types). This library fixes:
 *   - Philox4x32-10 (Salmon et al., SC 2011) with key = (lo, hi) words of
 *     seed.machine_id and counter = (lo(b), hi(b), seed.step, seed.sample_id)
 *     for block b = e >> 2 of global element index e; element e uses word
 *     e & 3 of its block;
 *   - Box-Muller on the word pairs (0,1) and (2,3) of a block:
 *     u_a = ((x_a >> 9) + 1/2) 2^-23, u_b = ((x_b >> 8) + 1/2) 2^-24,
 *     r = sqrt(-2 ln u_a); even element r cos(2 pi u_b), odd r sin(2 pi u_b).
 *   z depends only on (seed, e): never on the tensor split, the launch
 *   geometry or the GPU run, so every replica regenerates identical noise.
 *   Scope of that bit-identity: the Philox words are exact integers and the
 *   same on any machine; the transform is fp32 with every rounding explicit,
 *   except its reciprocal and square root, which are the GPU's
 *   rcp.approx / sqrt.approx instructions. z is therefore bitwise identical
 *   on every sm_103a (GB300) GPU, the only target of this library; on other
 *   hardware its last bits may differ, while staying within 1e-6 of the exact
 *   definition above.
 *
 * Global element index. Each tensor ("segment") carries flat_offset, the
 * global index of its element 0: element i of the segment is e = flat_offset
 * + i. Every replica must use the same table (part of the shared model
 * layout). Recommended: flat_offset of tensor t = align_up(flat_offset of
 * t-1 + numel of t-1, 8) in named_parameters() order. The vectorised path
 * needs (ptr - flat_offset * sizeof(T)) to be a multiple of 16 bytes; other
 * segments are still handled, element by element, at lower speed.
 *
 * Arithmetic. z = s r in fp32, with r the radius and s the signed cosine or
 * sine of the element; |z| <= sqrt(48 ln 2) = 5.77. A scaled draw a z is formed
 * as fma(s, a r, .) with a r rounded once to fp32. Perturb: theta + eps z as
 * one fp32 fused multiply-add, fma(s, eps r, theta), then one rounding to the
 * storage type (nearest, ties to even). Update: acc = 0; for each pair k in
 * canonical order acc = fma(s_k, c_k r_k, acc) in fp32; theta <- round(theta +
 * acc) once. No flush-to-zero. Results are bitwise repeatable.
 *
 * Memory and streams. The caller owns all device memory (e.g. torch
 * tensors). The library copies the host arrays it is given (segments, seeds,
 * codes) during the call, keeps no pointer to them, allocates no device
 * memory and holds no state between calls other than a per-device cache of
 * the SM count. Work is enqueued on `stream` (a cudaStream_t; NULL is the
 * legacy default stream) and the call returns without waiting for it. Calls on
 * different streams that touch the same parameters race.
 *
 * Errors. Every entry point returns a jb_status. Argument errors are detected
 * before anything is enqueued, and then nothing is enqueued. JB_ERR_CUDA
 * reports a failed CUDA runtime call or launch of this call (cudaGetLastError);
 * faults during execution surface at the caller's next synchronisation. The
 * library links the CUDA runtime statically, so its error state is private: an
 * error pending in the caller's runtime (torch's, say) is neither reported nor
 * cleared by libjb, and libjb clears each error it reports so that none lingers
 * into a later call. A sticky error (a fault that poisons the context) is
 * reported by every runtime. No exception, abort or exit crosses this
 * interface.
 */
#ifndef JB_H
#define JB_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* cudaStream_t is struct CUstream_st* */

typedef enum {
    JB_OK = 0,
    JB_ERR_INVALID_ARG = -1,      /* NULL pointer, negative count, bad scalar, overlap */
    JB_ERR_UNSUPPORTED_DTYPE = -2,
    JB_ERR_MISALIGNED = -3,       /* segment pointer not aligned to its element size */
    JB_ERR_DUPLICATE_SEED = -4,   /* two pairs with the same (machine_id, step, sample_id) */
    JB_ERR_CUDA = -5,             /* a CUDA runtime call or launch failed */
    JB_ERR_RANGE = -6,            /* a coefficient -lr deq(q) / denom is not finite in fp32 */
    JB_ERR_TOO_MANY_SEEDS = -7,   /* K above jb_max_seeds_per_call() */
    JB_ERR_NO_MEMORY = -8         /* host memory for the call's working copy could not be had */
} jb_status;

typedef enum { JB_F32 = 0, JB_BF16 = 1 } jb_dtype;

/* One parameter tensor: `numel` contiguous elements of the call's dtype at
 * device address `ptr` (caller-owned), element i having global index
 * flat_offset + i. Segments must not overlap in memory nor in global index. */
typedef struct {
    void* ptr;
    uint64_t numel;
    uint64_t flat_offset;
} jb_segment;

/* Seed s of Algorithm 1: the machine's start time (as an identifier), the
 * iteration, and the sample's index within the iteration. 16 bytes. */
typedef struct {
    uint64_t machine_id;
    uint32_t step;
    uint32_t sample_id;
} jb_seed;

/*
 * jb_perturb -- PerturbParameters(theta, eps, s) (Algorithm 1, subroutine):
 * for every element e of every segment, theta_e <- round_T(theta_e + eps
 * z_e(seed)), the sum one fp32 fused multiply-add (see Arithmetic). In place,
 * asynchronous on `stream`.
 *   segs, n_segs  segment table (host array, copied); n_segs = 0 is a no-op.
 *   dtype         JB_F32 or JB_BF16 for all segments.
 *   eps           finite perturbation scale (use +eps, -2 eps, +eps for one
 *                 SPSA sample; eps = 0 still rewrites theta unchanged).
 */
int jb_perturb(const jb_segment* segs, int n_segs, int dtype, jb_seed seed, float eps,
               struct CUstream_st* stream);

/*
 * jb_apply_updates -- apply K machines' projected gradients in one pass
 * (Section 2; Algorithm 1, gradient application):
 *   theta_e <- round_T(theta_e + sum_k c_k z_e(seeds[k])),
 *   c_k = (float)(-(double)lr * deq(q[k]) / (double)denom) with deq as in
 *   jb_dequantize_grad, pairs taken in ascending (machine_id, step,
 *   sample_id) order whatever order they are passed in.
 * The paper divides by the number of collected gradients (denom = K);
 * Section 4 scales the learning rate with sqrt(#perturbations): denom is
 * therefore the caller's.
 *   seeds, q, K   host arrays of K pairs (copied). K = 0 is a no-op.
 *                 K <= jb_max_seeds_per_call(); duplicates are an error.
 *   lr, denom     finite, denom != 0. qscale: S > 0 of the byte code.
 * Returns JB_ERR_RANGE (nothing enqueued) if some c_k is not finite in fp32.
 */
int jb_apply_updates(const jb_segment* segs, int n_segs, int dtype, const jb_seed* seeds,
                     const int8_t* q, int K, float lr, float denom, float qscale,
                     struct CUstream_st* stream);

/*
 * jb_apply_updates_from -- the step update applied to the weight backup, fused
 * with the restore (Algorithm 1: theta is reset from the backup copy, then every
 * machine's gradients; Section 2: the backup avoids the drift of theta + z - z):
 *   dst_e <- round_T(src_e + sum_k c_k z_e(seeds[k])), one read of src and one
 *   write of dst per element (and one more write of src when write_src != 0, so
 *   the next iteration's backup is refreshed in the same pass).
 * Same pairs, coefficients, canonical order and rounding as jb_apply_updates;
 * K = 0 copies src to dst.
 *   src, dst   tables of n_segs segments: dst[i] has the numel and flat_offset of
 *              src[i]; dst[i] is either src[i] itself or overlaps no source and
 *              no other destination.
 */
int jb_apply_updates_from(const jb_segment* src, const jb_segment* dst, int n_segs, int dtype,
                          const jb_seed* seeds, const int8_t* q, int K, float lr, float denom,
                          float qscale, int write_src, struct CUstream_st* stream);

/*
 * jb_replay_updates -- a late joiner's catch-up (Appendix B): after downloading
 * the weights, apply the projected gradients of every iteration it missed. Step
 * t holds step_sizes[t] pairs (consecutive in seeds/q) and its own lr[t] and
 * denom[t]; steps are applied in order, each rounded to the storage type as
 * jb_apply_updates would round it, so the result is bitwise that of n_steps
 * successive jb_apply_updates calls -- but theta is read and written once per
 * launch instead of once per step. A step holds at most
 * jb_max_seeds_per_call() pairs; steps are packed into launches of at most
 * that many pairs.
 */
int jb_replay_updates(const jb_segment* segs, int n_segs, int dtype, const jb_seed* seeds,
                      const int8_t* q, const int* step_sizes, int n_steps, const float* lr,
                      const float* denom, float qscale, struct CUstream_st* stream);

/* A tensor of 4-bit weights: numel codes, two per byte (element 2i in the low
 * nibble of byte i; `codes` 8-byte aligned, (numel + 1) / 2 bytes), and one fp32
 * scale per block of 64 elements (`scale`, ceil(numel / 64) floats). Weight i
 * is level[code_i] * scale[i / 64] with the 16 levels of jb_q4_levels().
 * flat_offset (a multiple of 4) is the global index of element 0, as for
 * jb_segment. Device memory, caller-owned. */
typedef struct {
    uint8_t* codes;
    float* scale;
    uint64_t numel;
    uint64_t flat_offset;
} jb_q4_segment;

/*
 * jb_perturb_q4 -- PerturbParameters on 4-bit weights (Section 3, Training
 * Speed: weights are dequantized before the noise is added and quantized
 * again). For every block of 64 elements: w_i = level[code_i] * scale,
 * w'_i = w_i + eps z_i(seed) in fp32, one fused multiply-add as in jb_perturb, then
 * scale' = max_i |w'_i| and code'_i = the nearest level to w'_i / scale' (ties
 * to the lower level; scale' = 0 gives the zero level). Codes and scales are
 * rewritten in place, asynchronously on `stream`; an odd numel leaves the
 * unused high nibble of the last byte as it was. The paper fixes no 4-bit
 * format; this is a NormalFloat-style code after QLoRA (see jb_q4_levels).
 * Errors, found before anything is enqueued: JB_ERR_INVALID_ARG for n_segs < 0,
 * a null array or pointer, a non-finite eps, an index range past 2^62, or
 * tensors whose bytes or index ranges overlap; JB_ERR_MISALIGNED for codes not
 * 8-byte aligned, scale not 4-byte aligned or flat_offset not a multiple of 4.
 * Tensors with numel = 0 are skipped.
 */
int jb_perturb_q4(const jb_q4_segment* segs, int n_segs, jb_seed seed, float eps,
                  struct CUstream_st* stream);

/* The 16 levels of the 4-bit code, ascending, in [-1, 1]: quantiles of N(0,1)
 * at probabilities d + (1/2 - d) j / 7 (j = 0..7, the median 0 last) and
 * 1/2 + (1/2 - d) j / 8 (j = 1..8), d = 1/32, divided by the largest, rounded
 * to fp32. Host only; out receives 16 floats. */
int jb_q4_levels(float* out);

/*
 * jb_checksum -- hash of the model for ChecksumMatch (Algorithm 1: each machine
 * checks with a random peer that their hashed theta match). The paper fixes no
 * hash. This one: cut the global element index space into 16-byte windows of
 * storage (8 bf16 or 4 fp32 elements; window v = elements [vE, vE + E)). For
 * every segment and every window v it overlaps, take the window's four 32-bit
 * storage words (little-endian; elements outside the segment read as 0), apply
 * the first four Philox4x32 rounds under key (lo32(v) ^ 0x6A09E667,
 * hi32(v) ^ 0xF3BCC908), and add (x1:x0) + (x3:x2). The checksum is the sum
 * mod 2^64. It depends on the values, the dtype and the flat offsets, not on
 * the launch; replicas with the same table and bits get the same value.
 *   d_out   device pointer to one uint64_t (8-byte aligned, caller-owned); it is
 *           zeroed and written on `stream`.
 */
int jb_checksum(const jb_segment* segs, int n_segs, int dtype, uint64_t* d_out,
                struct CUstream_st* stream);

/*
 * jb_quantize_grad -- one-byte projected gradient (Section 3, Training
 * Speed: the sign and the logarithm of the magnitude, limited to +-127). Host
 * only, pure:
 *   *out = sign(g) * min(127, round_half_away(qscale * ln(1 + |g|))),
 *   NaN -> 0, +-inf -> +-127. qscale must be finite and > 0.
 */
int jb_quantize_grad(double g, float qscale, int8_t* out);

/*
 * jb_dequantize_grad -- inverse of the byte code, host only, pure:
 *   *out = (float)(sign(q) * expm1(min(|q|, 127) / qscale)) (code -128 reads as
 *   -127). Computed in double, rounded once; may be +-inf for small qscale.
 */
int jb_dequantize_grad(int8_t q, float qscale, float* out);

/* Largest K accepted by jb_apply_updates in one call (the pairs travel in the
 * kernel's parameter space). */
int jb_max_seeds_per_call(void);

/* Static description of a status code. Never NULL. */
const char* jb_status_string(int status);

/* ---------------------------------------------------------------------------
 * Test hooks (not on the hot path). Device buffers are caller-owned.
 * ------------------------------------------------------------------------- */

/* d_out[4 i + w] = word w of Philox block first_block + i under `seed`.
 * d_out must be 16-byte aligned (JB_ERR_MISALIGNED); n_blocks <= 2^38. */
int jb_debug_philox(jb_seed seed, uint64_t first_block, uint64_t n_blocks, uint32_t* d_out,
                    struct CUstream_st* stream);

/* *d_out = XOR of all words of Philox blocks first_block .. first_block +
 * n_blocks - 1 under `seed`: the generator alone, computed as the kernels
 * compute it, on the persistent grid (the benchmark times it as the
 * generator-only rate). d_out: one uint32_t, 4-byte aligned, zeroed and written
 * on `stream`. n_blocks <= 2^46, first_block <= 2^60. */
int jb_debug_philox_fold(jb_seed seed, uint64_t first_block, uint64_t n_blocks, uint32_t* d_out,
                         struct CUstream_st* stream);

/* d_out[i] = z of global element first_elem + i under `seed` (fp32).
 * d_out must be 4-byte aligned (JB_ERR_MISALIGNED); n <= 2^38. */
int jb_debug_gaussian(jb_seed seed, uint64_t first_elem, uint64_t n, float* d_out,
                      struct CUstream_st* stream);

/* Box-Muller of raw word pairs: d_out[2 i], d_out[2 i + 1] = z of the even and
 * odd element for words (d_words[2 i], d_words[2 i + 1]). Both buffers must be
 * 4-byte aligned (JB_ERR_MISALIGNED); n_pairs <= 2^38. */
int jb_debug_box_muller(const uint32_t* d_words, uint64_t n_pairs, float* d_out,
                        struct CUstream_st* stream);

/* jb_checksum / jb_perturb / jb_apply_updates with an explicit number of CTAs
 * (0 = the default persistent grid); results must not depend on it. */
int jb_checksum_with_grid(const jb_segment* segs, int n_segs, int dtype, uint64_t* d_out,
                          int grid_ctas, struct CUstream_st* stream);
int jb_perturb_with_grid(const jb_segment* segs, int n_segs, int dtype, jb_seed seed, float eps,
                         int grid_ctas, struct CUstream_st* stream);
int jb_apply_updates_with_grid(const jb_segment* segs, int n_segs, int dtype,
                               const jb_seed* seeds, const int8_t* q, int K, float lr,
                               float denom, float qscale, int grid_ctas,
                               struct CUstream_st* stream);

#ifdef __cplusplus
}
#endif
#endif /* JB_H */
