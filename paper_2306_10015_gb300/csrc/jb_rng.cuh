// jb_rng.cuh -- the seeded N(0,1) stream, computed in registers on sm_103a.
//
// PerturbParameters (Algorithm 1, subroutine) reseeds a generator with
// s = (machine time id, iteration, sample index) and draws z ~ N(0,1) for every
// parameter. Here z of global element e is a pure function of (s, e):
//   Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC 2011) of counter
//   (lo(b), hi(b), step, sample_id), b = e >> 2, under key (lo(mid), hi(mid));
//   Box-Muller (Box & Muller 1958) on word pairs (0,1) and (2,3):
//   r = sqrt(-2 ln u_a), u_a = ((x_a >> 9) + 1/2) 2^-23; angle 2 pi u_b,
//   u_b = ((x_b >> 8) + 1/2) 2^-24; element 4b + 2p -> r cos, 4b + 2p + 1 -> r sin.
// Nothing here is written to memory on the hot path.
#pragma once
#include <cstdint>

namespace jb {

// Philox4x32 round multipliers and key increments (Salmon et al. 2011).
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

struct Key {
    uint32_t k0, k1;       // machine id, low and high word
    uint32_t step, sample; // counter words 2 and 3
};

// One Philox round on (x0, x1, x2, x3) with round key (k0, k1).
__device__ __forceinline__ void philox_round(uint32_t& x0, uint32_t& x1, uint32_t& x2,
                                             uint32_t& x3, uint32_t k0, uint32_t k1) {
    const uint64_t p0 = static_cast<uint64_t>(kPhiloxM0) * x0;
    const uint64_t p1 = static_cast<uint64_t>(kPhiloxM1) * x2;
    const uint32_t y0 = static_cast<uint32_t>(p1 >> 32) ^ x1 ^ k0;
    const uint32_t y2 = static_cast<uint32_t>(p0 >> 32) ^ x3 ^ k1;
    x1 = static_cast<uint32_t>(p1);
    x3 = static_cast<uint32_t>(p0);
    x0 = y0;
    x2 = y2;
}

// Four words of Philox4x32-10 block (b_lo, b_hi) under key.
__device__ __forceinline__ uint4 philox_block(const Key& key, uint32_t b_lo, uint32_t b_hi) {
    uint32_t x0 = b_lo, x1 = b_hi, x2 = key.step, x3 = key.sample;
    uint32_t k0 = key.k0, k1 = key.k1;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        philox_round(x0, x1, x2, x3, k0, k1);
        k0 += kPhiloxW0;
        k1 += kPhiloxW1;
    }
    return make_uint4(x0, x1, x2, x3);
}

// Box-Muller of one word pair: (r cos 2 pi u_b, r sin 2 pi u_b).
// u_a = (2 (x_a >> 9) + 1) 2^-24 is exact in fp32. The angle 2 pi u_b = pi t
// with t = (2 (x_b >> 8) + 1) 2^-24 in (0, 2); the half turn is taken out
// exactly from the top bit (sin and cos change sign), leaving t in (0, 1) with
// a 24-bit odd numerator, also exact in fp32.
__device__ __forceinline__ float2 box_muller(uint32_t xa, uint32_t xb) {
    const float ua = __uint2float_rn(((xa >> 9) << 1) | 1u) * 0x1p-24f;
    const float r = sqrtf(-2.0f * logf(ua));
    const uint32_t mb = xb >> 8;
    const float t = __uint2float_rn(((mb & 0x7FFFFFu) << 1) | 1u) * 0x1p-24f;
    float s, c;
    sincospif(t, &s, &c);
    const uint32_t flip = (mb & 0x800000u) << 8;  // sign bit when t was in [1, 2)
    s = __uint_as_float(__float_as_uint(s) ^ flip);
    c = __uint_as_float(__float_as_uint(c) ^ flip);
    return make_float2(__fmul_rn(r, c), __fmul_rn(r, s));
}

// The four Gaussians of block (b_lo, b_hi), elements 4b .. 4b + 3.
__device__ __forceinline__ float4 block_gaussians(const Key& key, uint32_t b_lo, uint32_t b_hi) {
    const uint4 w = philox_block(key, b_lo, b_hi);
    const float2 z01 = box_muller(w.x, w.y);
    const float2 z23 = box_muller(w.z, w.w);
    return make_float4(z01.x, z01.y, z23.x, z23.y);
}

}  // namespace jb
