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
// A lane takes 32 consecutive elements, so a 64-element block is two lanes and
// its maximum is one butterfly shuffle.
//
// Dequantizing reads two levels at once: the codes of elements 4b and 4b + 2 are
// nibbles 0 and 2 of a 16-bit group (4b + 1 and 4b + 3: nibbles 1 and 3), and a
// shared-memory table holds (level[a], level[b]) at byte offset 8 a + 2048 b, so
// one shift and one mask of the code word give the address of both.
//
// Nearest level = the number of midpoints strictly below x. Consecutive
// midpoints are more than 1/16 apart, so each bucket [j/16, (j+1)/16) of
// [-1, 1) holds at most one; with b = floor(16 x) (exact in fp32), the code is
// (midpoints below the bucket) + (x > the bucket's midpoint, if any): one
// shared-memory read and one comparison instead of a 4-step binary search.
#include <cuda_bf16.h>

#include <atomic>

#include "jb_internal.h"
#include "jb_q4.h"
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

// Buckets: bucket[j] for j < 32 = (the midpoint in [(j - 16)/16, (j - 15)/16) or
// +inf, the number of midpoints below (j - 16)/16 as integer bits); bucket[32 .. 63]
// = (+inf, 15), for x = 1. For x in [-1, 1], y = x 2^-16 + 1 + 2^-16 rounded toward
// minus infinity lies in [1, 1 + 2^-15], and its fraction bits 3 .. 8 are
// floor(16 (x + 1)): the exact value is 1 + 128 (x + 1) 2^-23, every multiple of
// 2^-20 there is representable, so rounding down never crosses one. The mask gives
// the byte offset of the 8-byte entry directly; a NaN x gets an unspecified code.
constexpr float kQ4IdxBias = 0x1.0001p+0f;  // 1 + 2^-16

__device__ __forceinline__ uint32_t q4_code(float x, float y, const float2* bucket) {
    const uint32_t off = __float_as_uint(y) & 0x1F8u;
    const float2 e = *reinterpret_cast<const float2*>(reinterpret_cast<const char*>(bucket) + off);
    return __float_as_uint(e.y) + (x > e.x ? 1u : 0u);
}

// max(a, b, c) in one instruction
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// (level[a], level[b]) at byte offset 8 a + 2048 b: 15 * 256 + 16 entries, 256 used
constexpr int kPairEntries = 15 * 256 + 16;

// Levels of the codes in nibbles (n, n + 2) of cw, n = 4 BB + (ODD ? 1 : 0):
// elements (4b, 4b + 2) or (4b + 1, 4b + 3) of the word's block b = BB.
template <int BB, bool ODD>
__device__ __forceinline__ float2 pair_at(const float2* pair, uint32_t cw) {
    constexpr int sh = 16 * BB + (ODD ? 4 : 0) - 3;
    const uint32_t off = (sh < 0 ? cw << (-sh) : cw >> sh) & 0x7878u;
    return *reinterpret_cast<const float2*>(reinterpret_cast<const char*>(pair) + off);
}

template <int B>
__device__ __forceinline__ void dequant_block(const float2* pair, const uint32_t* cw, float2& le, float2& lo) {
    le = pair_at<B % 2, false>(pair, cw[B / 2]);
    lo = pair_at<B % 2, true>(pair, cw[B / 2]);
}

constexpr int kThreadsQ4 = 512;

// 64 registers: two CTAs per SM (8 bytes spilled), measured 2.7% faster than the
// compiler's 70 registers and one CTA
__global__ void __maxnreg__(64) q4_perturb_kernel(const __grid_constant__ Q4Params p) {
    constexpr int E = kQ4Epl, NB = E / 4, NW = E / 8;
    static_assert(kQ4UnitsPerBlock == 2 && NB == 8, "two 32-element lanes per block");
    __shared__ float2 pair[kPairEntries];
    __shared__ float2 bucket[64];
    for (int i = threadIdx.x; i < 256; i += kThreadsQ4)
        pair[(i & 15) + 256 * (i >> 4)] = make_float2(c_level[i & 15], c_level[i >> 4]);
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
    const float2 eps2 = splat(p.seed.coef);
    uint32_t s = 0;
    // all 32 lanes run every iteration (the block maximum is a warp shuffle)
    for (uint64_t wt = warp; wt * 32u < p.n_units; wt += n_warps) {
        const uint64_t unit = wt * 32u + lane;
        const bool valid = unit < p.n_units;
        if (valid)
            while (s + 1 < p.n_segs && p.segs[s + 1].unit0 <= unit) ++s;
        const SegParamQ4& g = p.segs[s];
        const uint64_t u = unit - g.unit0;
        const int64_t i0 = static_cast<int64_t>(E * u);
        const int64_t n = static_cast<int64_t>(g.n);
        const bool any = valid && i0 < n;
        const bool full = valid && i0 + E <= n;
        uint8_t* codes = reinterpret_cast<uint8_t*>(g.codes);
        float* scale = reinterpret_cast<float*>(g.scale);

        uint32_t cw[NW];  // 32 codes, 8 per word
#pragma unroll
        for (int j = 0; j < NW; ++j) cw[j] = 0u;
        if (full) {
#pragma unroll
            for (int j = 0; j < NW; j += 2) {  // codes are 8-byte aligned
                const uint2 v = *reinterpret_cast<const uint2*>(codes + i0 / 2 + 4 * j);
                cw[j] = v.x;
                cw[j + 1] = v.y;
            }
        } else if (any) {
#pragma unroll
            for (int b = 0; b < E / 2; ++b)
                if (i0 + 2 * b < n) cw[b / 4] |= static_cast<uint32_t>(codes[i0 / 2 + b]) << (8 * (b % 4));
        }
        const float2 s2 = splat(any ? scale[u >> 1] : 0.0f);

        // dequantize and perturb: w = fma(cos or sin, eps r, level * scale), the
        // Philox words of block b + 1 computed while block b is transformed;
        // wv[2b] = elements (4b, 4b + 2), wv[2b + 1] = (4b + 1, 4b + 3)
        float2 wv[E / 2];
        const uint64_t blk0 = (g.fo + static_cast<uint64_t>(i0)) >> 2;  // fo % 4 == 0
        uint4 wcur = philox_block(sc, static_cast<uint32_t>(blk0), static_cast<uint32_t>(blk0 >> 32));
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            uint4 wnext;
            if (b + 1 < NB)
                wnext = philox_block(sc, static_cast<uint32_t>(blk0 + b + 1),
                                     static_cast<uint32_t>((blk0 + b + 1) >> 32));
            const Polar2 o = polar2(wcur);
            if (b + 1 < NB) wcur = wnext;
            const float2 rc = mul2<kPackO>(eps2, o.rr);
            float2 le, lo;
            switch (b) {
                case 0: dequant_block<0>(pair, cw, le, lo); break;
                case 1: dequant_block<1>(pair, cw, le, lo); break;
                case 2: dequant_block<2>(pair, cw, le, lo); break;
                case 3: dequant_block<3>(pair, cw, le, lo); break;
                case 4: dequant_block<4>(pair, cw, le, lo); break;
                case 5: dequant_block<5>(pair, cw, le, lo); break;
                case 6: dequant_block<6>(pair, cw, le, lo); break;
                default: dequant_block<7>(pair, cw, le, lo); break;
            }
            wv[2 * b] = fma2<kPackO>(o.cm, rc, mul2<true>(le, s2));
            wv[2 * b + 1] = fma2<kPackO>(o.sm, rc, mul2<true>(lo, s2));
        }
        // elements past the end of the segment do not count towards the maximum
        if (!full) {
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                if (i0 + 4 * b + 0 >= n) wv[2 * b].x = 0.0f;
                if (i0 + 4 * b + 2 >= n) wv[2 * b].y = 0.0f;
                if (i0 + 4 * b + 1 >= n) wv[2 * b + 1].x = 0.0f;
                if (i0 + 4 * b + 3 >= n) wv[2 * b + 1].y = 0.0f;
            }
        }
        float m = 0.0f;
#pragma unroll
        for (int i = 0; i < E / 2; ++i) m = fmax3(m, fabsf(wv[i].x), fabsf(wv[i].y));
        // block maximum over the two lanes of the block (lanes 2j, 2j + 1)
        m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 1));
        // 1/m rounded down: every |w / m| then rounds to at most 1, so x needs no clamp
        const float2 inv2 = splat(m > 0.0f ? __frcp_rd(m) : 0.0f);

        // quantize again: x = w / m, its bucket from y = RD(x 2^-16 + 1 + 2^-16)
        uint32_t ow[NW];
#pragma unroll
        for (int j = 0; j < NW; ++j) ow[j] = 0u;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const float2 x = mul2<true>(wv[2 * b + h], inv2);
                const float2 y = __ffma2_rd(x, splat(0x1p-16f), splat(kQ4IdxBias));
                const int ka = 4 * b + h, kb = 4 * b + h + 2;
                ow[ka / 8] += q4_code(x.x, y.x, bucket) << (4 * (ka % 8));
                ow[kb / 8] += q4_code(x.y, y.y, bucket) << (4 * (kb % 8));
            }
        }
        if (full) {
#pragma unroll
            for (int j = 0; j < NW; j += 2)
                *reinterpret_cast<uint2*>(codes + i0 / 2 + 4 * j) = make_uint2(ow[j], ow[j + 1]);
        } else if (any) {
#pragma unroll
            for (int b = 0; b < E / 2; ++b) {
                if (i0 + 2 * b >= n) continue;
                const uint8_t byte = static_cast<uint8_t>(ow[b / 4] >> (8 * (b % 4)));
                // an odd tail leaves the unused high nibble of the last byte as it was
                codes[i0 / 2 + b] = (i0 + 2 * b + 1 < n) ? byte
                                                         : static_cast<uint8_t>((codes[i0 / 2 + b] & 0xF0u) | (byte & 0x0Fu));
            }
        }
        if (any && (u & 1u) == 0u) scale[u >> 1] = m;
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
