// jb_q4.cu -- PerturbParameters on 4-bit weights (Section 3, Training Speed:
// layer weights are dequantized before the noise is added and quantized again).
//
// Code (the paper fixes none; it cites QLoRA's NormalFloat): 16 levels built
// from quantiles of N(0,1) and scaled to [-1, 1] (gen_q4_levels.py); blocks of
// 64 elements share one fp32 scale, the largest |w| of the block; a weight is
// level[code] * scale; quantizing picks the nearest level (ties to the lower).
//
// Per element: dequantize, w' = w + eps z as one fused multiply-add (as in the
// plain perturbation) with the same z as every other path (global index
// flat_offset + i), then per block scale' = max |w'| and
// code' = nearest level of w' / scale'. Codes and scales are rewritten in place.
// A 64-element block is four consecutive lanes (16 elements each): its maximum
// is two butterfly shuffles. Levels live in shared memory, read with
// data-dependent indices (16 distinct words: no bank conflicts).
//
// Nearest level = the number of midpoints strictly below x. Consecutive
// midpoints are more than 1/16 apart, so each bucket [j/16, (j+1)/16) of
// [-1, 1) holds at most one; with b = floor(16 x) (exact in fp32), the code is
// (midpoints below the bucket) + (x > the bucket's midpoint, if any): one
// shared-memory read and one comparison instead of a 4-step binary search.
#include <cuda_bf16.h>

#include <atomic>

#include "jb_internal.h"
#include "jb_rng.cuh"

namespace jb {
namespace {

// gen_q4_levels.py
constexpr float kQ4Level[16] = {
    -0x1.000000p+0f, -0x1.6311acp-1f, -0x1.0b8d60p-1f, -0x1.924c0ap-2f, -0x1.21b102p-2f,
    -0x1.7851c6p-3f, -0x1.72d976p-4f, 0x0.0p+0f,       0x1.4421acp-4f,  0x1.47c076p-3f,
    0x1.f54804p-3f,  0x1.582f80p-2f,  0x1.c1002ap-2f,  0x1.1eba52p-1f,  0x1.70ca9ap-1f,
    0x1.000000p+0f};

__constant__ float c_level[16] = {
    kQ4Level[0], kQ4Level[1], kQ4Level[2],  kQ4Level[3],  kQ4Level[4],  kQ4Level[5],
    kQ4Level[6], kQ4Level[7], kQ4Level[8],  kQ4Level[9],  kQ4Level[10], kQ4Level[11],
    kQ4Level[12], kQ4Level[13], kQ4Level[14], kQ4Level[15]};
// midpoints (L_j + L_j+1) / 2 of the fp32 levels, rounded to fp32 (gen_q4_levels.py)
__constant__ float c_mid[15] = {
    -0x1.b188d6p-1f, -0x1.374f86p-1f, -0x1.d4b364p-2f, -0x1.59fe86p-2f, -0x1.ddd9e4p-3f,
    -0x1.18df40p-3f, -0x1.72d976p-5f, 0x1.4421acp-5f,  0x1.e9d14cp-4f,  0x1.9e843cp-3f,
    0x1.2969c0p-2f,  0x1.8c97d4p-2f,  0x1.ff3a68p-2f,  0x1.47c276p-1f,  0x1.b8654cp-1f};

// Nearest level of x in [-1, 1] (ties to the lower): the number of midpoints
// strictly below x. bucket[j] for j < 32 = (the midpoint in [(j - 16)/16,
// (j - 15)/16) or +inf, the number of midpoints below (j - 16)/16 as integer
// bits); bucket[32 .. 63] = (+inf, 15), for x = 1. The index floor(16 (x + 1))
// is read from the fraction bits of x / 2 + 5/2 rounded toward minus infinity:
// that value lies in [2, 3], where the fraction's top six bits are
// floor(16 (x + 1)), and rounding down never crosses a multiple of 1/32 (all of
// them are representable there). The shift and mask give the byte offset of the
// 8-byte entry directly; a NaN x gets an unspecified code.
__device__ __forceinline__ uint32_t q4_code(float x, const float2* bucket) {
    const uint32_t off = (__float_as_uint(__fmaf_rd(x, 0.5f, 2.5f)) >> 14) & 0x1F8u;
    const float2 e = *reinterpret_cast<const float2*>(reinterpret_cast<const char*>(bucket) + off);
    return __float_as_uint(e.y) + (x > e.x ? 1u : 0u);
}

// level[code j of the word cw]: the code's byte offset in the table (4 code) is
// taken from the word directly, one shift and one mask.
__device__ __forceinline__ float level_at(const float* level, uint32_t cw, int j) {
    const uint32_t off = (j == 0 ? cw << 2 : cw >> (4 * j - 2)) & 0x3Cu;
    return *reinterpret_cast<const float*>(reinterpret_cast<const char*>(level) + off);
}

constexpr int kThreadsQ4 = 512;  // measured 2.4% faster than 256 on the 13B-shaped set

__global__ void __launch_bounds__(kThreadsQ4) q4_perturb_kernel(const __grid_constant__ Q4Params p) {
    __shared__ float level[16];
    __shared__ float2 bucket[64];
    if (threadIdx.x < 16) level[threadIdx.x] = c_level[threadIdx.x];
    if (threadIdx.x >= 32 && threadIdx.x < 64)
        bucket[threadIdx.x] = make_float2(__int_as_float(0x7F800000), __uint_as_float(15u));
    if (threadIdx.x < 32) {
        const float lo = static_cast<float>(static_cast<int>(threadIdx.x) - 16) * 0.0625f;
        const float hi = lo + 0.0625f;
        uint32_t below = 0;
        float m = __int_as_float(0x7F800000);  // +inf: no midpoint in the bucket
#pragma unroll
        for (int k = 0; k < 15; ++k) {
            const float md = c_mid[k];
            below += md < lo ? 1u : 0u;
            if (md >= lo && md < hi) m = md;
        }
        bucket[threadIdx.x] = make_float2(m, __uint_as_float(below));
    }
    __syncthreads();  // every thread reaches this before any work

    const uint32_t lane = threadIdx.x & 31u;
    const uint64_t warp = (static_cast<uint64_t>(blockIdx.x) * kThreadsQ4 + threadIdx.x) >> 5;
    const uint64_t n_warps = (static_cast<uint64_t>(gridDim.x) * kThreadsQ4) >> 5;
    const SeedConst sc = seed_const(Key{p.seed.k0, p.seed.k1, p.seed.step, p.seed.sample});
    const float eps = p.seed.coef;
    uint32_t s = 0;
    // all 32 lanes run every iteration (the block maximum is a warp shuffle)
    for (uint64_t wt = warp; wt * 32u < p.n_units; wt += n_warps) {
        const uint64_t unit = wt * 32u + lane;
        const bool valid = unit < p.n_units;
        if (valid)
            while (s + 1 < p.n_segs && p.segs[s + 1].unit0 <= unit) ++s;
        const SegParamQ4& g = p.segs[s];
        const uint64_t u = unit - g.unit0;
        const int64_t i0 = static_cast<int64_t>(16 * u);
        const int64_t n = static_cast<int64_t>(g.n);
        const bool any = valid && i0 < n;
        const bool full = valid && i0 + 16 <= n;
        uint8_t* codes = reinterpret_cast<uint8_t*>(g.codes);
        float* scale = reinterpret_cast<float*>(g.scale);

        uint32_t cw[2] = {0u, 0u};  // 16 codes
        if (full) {
            const uint2 v = *reinterpret_cast<const uint2*>(codes + i0 / 2);
            cw[0] = v.x;
            cw[1] = v.y;
        } else if (any) {
#pragma unroll
            for (int b = 0; b < 8; ++b)
                if (i0 + 2 * b < n) cw[b / 4] |= static_cast<uint32_t>(codes[i0 / 2 + b]) << (8 * (b % 4));
        }
        const float sc_in = any ? scale[u >> 2] : 0.0f;

        // dequantize and perturb: w = fma(cos or sin, eps r, level * scale), the
        // Philox words of block b + 1 computed while block b is transformed
        float w[16];
        const uint64_t blk0 = (g.fo + static_cast<uint64_t>(i0)) >> 2;  // fo % 4 == 0
        const float2 eps2 = splat(eps);
        uint4 wcur = philox_block(sc, static_cast<uint32_t>(blk0), static_cast<uint32_t>(blk0 >> 32));
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            uint4 wnext;
            if (b + 1 < 4)
                wnext = philox_block(sc, static_cast<uint32_t>(blk0 + b + 1),
                                     static_cast<uint32_t>((blk0 + b + 1) >> 32));
            const Polar2 o = polar2(wcur);
            if (b + 1 < 4) wcur = wnext;
            const float2 rc = mul2<kPackO>(eps2, o.rr);
            float lv[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const int k = 4 * b + t;
                lv[t] = __fmul_rn(level_at(level, cw[k / 8], k % 8), sc_in);
            }
            const float2 ev = fma2<kPackO>(o.cm, rc, make_float2(lv[0], lv[2]));
            const float2 od = fma2<kPackO>(o.sm, rc, make_float2(lv[1], lv[3]));
            w[4 * b + 0] = ev.x;
            w[4 * b + 1] = od.x;
            w[4 * b + 2] = ev.y;
            w[4 * b + 3] = od.y;
        }
        // elements past the end of the segment do not count towards the maximum
        if (!full) {
#pragma unroll
            for (int k = 0; k < 16; ++k)
                if (i0 + k >= n) w[k] = 0.0f;
        }
        float m = 0.0f;
#pragma unroll
        for (int k = 0; k < 16; ++k) m = fmaxf(m, fabsf(w[k]));
        // block maximum over the four lanes of the block (lanes 4j .. 4j + 3)
        m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 1));
        m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 2));
        // 1/m rounded down: every |w / m| then rounds to at most 1, so x needs no clamp
        const float inv = m > 0.0f ? __frcp_rd(m) : 0.0f;

        // quantize again
        uint32_t ow[2] = {0u, 0u};
#pragma unroll
        for (int k = 0; k < 16; ++k) ow[k / 8] += q4_code(__fmul_rn(w[k], inv), bucket) << (4 * (k % 8));
        if (full) {
            *reinterpret_cast<uint2*>(codes + i0 / 2) = make_uint2(ow[0], ow[1]);
        } else if (any) {
#pragma unroll
            for (int b = 0; b < 8; ++b) {
                if (i0 + 2 * b >= n) continue;
                const uint8_t byte = static_cast<uint8_t>(ow[b / 4] >> (8 * (b % 4)));
                // an odd tail leaves the unused high nibble of the last byte as it was
                codes[i0 / 2 + b] = (i0 + 2 * b + 1 < n) ? byte
                                                         : static_cast<uint8_t>((codes[i0 / 2 + b] & 0xF0u) | (byte & 0x0Fu));
            }
        }
        if (any && (u & 3u) == 0u) scale[u >> 2] = m;
    }
}

std::atomic<int> g_q4_grid[64];

}  // namespace

void q4_levels_host(float out[16]) {
    for (int i = 0; i < 16; ++i) out[i] = kQ4Level[i];
}

cudaError_t launch_q4_perturb(const Q4Params& p, int grid_ctas, cudaStream_t stream) {
    if (p.n_units == 0) return cudaSuccess;
    int grid = grid_ctas;
    if (grid <= 0) {
        int dev = 0;
        cudaError_t err = cudaGetDevice(&dev);
        if (err != cudaSuccess) return err;
        grid = dev < 64 ? g_q4_grid[dev].load(std::memory_order_relaxed) : 0;
        if (grid <= 0) {
            int sms = 0, per_sm = 0;
            err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (err != cudaSuccess) return err;
            err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, q4_perturb_kernel,
                                                                kThreadsQ4, 0);
            if (err != cudaSuccess) return err;
            grid = sms * (per_sm > 0 ? per_sm : 1);
            if (dev < 64) g_q4_grid[dev].store(grid, std::memory_order_relaxed);
        }
        const uint64_t needed = (p.n_units + kThreadsQ4 - 1) / kThreadsQ4;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    q4_perturb_kernel<<<grid, kThreadsQ4, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace jb
