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
//
// Arithmetic of the transform (fp32, every rounding explicit):
//   radius  u_a = 2^e f exactly, f in [3/4, 3/2), t = f - 1 exact; with
//           q = -4t / (2 + t) (one rcp.approx), -2 ln(1 + t) = q + q w R(w),
//           w = q^2, R a degree-2 minimax polynomial; L = -2 e ln 2 - 2 ln(1+t)
//           with 2 ln 2 split hi + lo (Cody & Waite 1980) so e (2 ln 2)_hi is
//           exact; r = sqrt.approx(L) (relative error below 1.1e-7 over
//           every L the transform produces; one special-function operation
//           where rsqrt.approx and a Newton step took four packed FP ones).
//   angle   the 24-bit angle index splits into an octant (3 bits, handled
//           exactly by reflection, swap and sign flips) and a 21-bit offset
//           x in (0, 1) of the octant, sin(pi x / 4) and cos(pi x / 4) by
//           minimax polynomials of degree 7 and 8 (relative error < 0.6 ulp
//           for the sine, also near zero; 7.2e-8 for the cosine, which the
//           octant keeps above 0.7).
// Coefficients: fit_poly.py (Remez exchange). The transform is checked
// against a double-precision evaluation of the same definition over all
// radius words and all angle words (|dz| <= 1e-6).
#pragma once
#include <cstdint>

namespace jb {

// Philox4x32 round multipliers and key increments (Salmon et al. 2011).
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

// Polynomials (fit_poly.py).
constexpr float kLogR0 = 0x1.5555b4p-6f, kLogR1 = 0x1.992aaap-11f, kLogR2 = 0x1.36ec6ap-15f;
constexpr float kSinHi = 0x1.921fb6p-1f;   // pi/4 = hi + lo
constexpr float kSinLo = -0x1.777a5cp-26f;
constexpr float kSinS0 = -0x1.4abbbep-4f, kSinS1 = 0x1.465facp-9f, kSinS2 = -0x1.2db5cep-15f;
constexpr float kCosC0 = -0x1.3bd3ccp-2f, kCosC1 = 0x1.03c1b0p-6f, kCosC2 = -0x1.55b2b6p-12f,
                kCosC3 = 0x1.d4f7eep-19f;
constexpr float kTwoLn2Hi = -0x1.62e4p+0f;       // -(2 ln 2) to 16 bits
constexpr float kTwoLn2Lo = -0x1.7f7d1cp-19f;    // -(2 ln 2) - kTwoLn2Hi

struct Key {
    uint32_t k0, k1;       // machine id, low and high word
    uint32_t step, sample; // counter words 2 and 3
};

// Per-seed constants: the first round's product of counter word 2 (the step)
// is the same for every block of a seed.
struct SeedConst {
    uint32_t k0, k1;
    uint32_t a_hi, a_lo;  // M1 * step
    uint32_t c;           // sample ^ k1
};

__device__ __forceinline__ SeedConst seed_const(const Key& key) {
    const uint64_t a = static_cast<uint64_t>(kPhiloxM1) * key.step;
    SeedConst s;
    s.k0 = key.k0;
    s.k1 = key.k1;
    s.a_hi = static_cast<uint32_t>(a >> 32);
    s.a_lo = static_cast<uint32_t>(a);
    s.c = key.sample ^ key.k1;
    return s;
}

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

// The seed-independent part of round 1 for block (b_lo, b_hi): the product of
// counter word 0 (the block's low word) and its high word. Every seed of an update
// shares it.
struct BlockCtr {
    uint32_t p_hi, p_lo;  // M0 * b_lo
    uint32_t b_hi;
};

__device__ __forceinline__ BlockCtr block_ctr(uint32_t b_lo, uint32_t b_hi) {
    const uint64_t p0 = static_cast<uint64_t>(kPhiloxM0) * b_lo;
    BlockCtr c;
    c.p_hi = static_cast<uint32_t>(p0 >> 32);
    c.p_lo = static_cast<uint32_t>(p0);
    c.b_hi = b_hi;
    return c;
}

// Four words of Philox4x32-10 for block c under the seed's constants: round 1 from
// the per-seed and per-block products, rounds 2 .. 10 in full.
__device__ __forceinline__ uint4 philox_block(const SeedConst& s, const BlockCtr& c) {
    uint32_t x0 = s.a_hi ^ c.b_hi ^ s.k0;
    uint32_t x1 = s.a_lo;
    uint32_t x2 = c.p_hi ^ s.c;
    uint32_t x3 = c.p_lo;
    uint32_t k0 = s.k0, k1 = s.k1;
#pragma unroll
    for (int r = 1; r < 10; ++r) {
        k0 += kPhiloxW0;
        k1 += kPhiloxW1;
        philox_round(x0, x1, x2, x3, k0, k1);
    }
    return make_uint4(x0, x1, x2, x3);
}

// Four words of Philox4x32-10 block (b_lo, b_hi).
__device__ __forceinline__ uint4 philox_block(const SeedConst& s, uint32_t b_lo, uint32_t b_hi) {
    return philox_block(s, block_ctr(b_lo, b_hi));
}

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float sqrt_approx(float x) {
    float y;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float2 splat(float a) { return make_float2(a, a); }

// Two fp32 operations at once: one packed fp32x2 instruction, or two scalar ones.
// Both round each component once to nearest, so the results are identical; the
// choice only moves work between the FMA pipes (packed instructions share the
// pipe that also runs the integer multiplies of Philox).
template <bool PACK>
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    if constexpr (PACK) return __ffma2_rn(a, b, c);
    return make_float2(__fmaf_rn(a.x, b.x, c.x), __fmaf_rn(a.y, b.y, c.y));
}
template <bool PACK>
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    if constexpr (PACK) return __fmul2_rn(a, b);
    return make_float2(__fmul_rn(a.x, b.x), __fmul_rn(a.y, b.y));
}
template <bool PACK>
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    if constexpr (PACK) return __fadd2_rn(a, b);
    return make_float2(__fadd_rn(a.x, b.x), __fadd_rn(a.y, b.y));
}

#ifndef JB_PACK_RADIUS
#define JB_PACK_RADIUS 1
#endif
#ifndef JB_PACK_ANGLE
#define JB_PACK_ANGLE 1
#endif
#ifndef JB_PACK_OUT
#define JB_PACK_OUT 1
#endif
constexpr bool kPackR = JB_PACK_RADIUS, kPackA = JB_PACK_ANGLE, kPackO = JB_PACK_OUT;

// Box-Muller of the two word pairs of a Philox block, (w.x, w.y) and (w.z, w.w), in
// lockstep: every floating-point step is one packed fp32x2 instruction (two IEEE
// round-to-nearest operations per issue slot), integer steps stay per pair. The
// radius is carried with its sign flipped where a packed operation cannot negate an
// operand (q = 4t/(2+t), L = 2 e ln 2 + 2 ln(1+t) = ln u_a^-2 negated, -r) and
// the sign is restored in the final sign masks; round-to-nearest is odd-symmetric,
// so no rounding differs from the unflipped formulas.
// Polar form: rr = (-r of pair A, -r of pair B); cm, sm = the signed cosines and sines
// (sign flips of the negated radius included), so z_even = cm rr, z_odd = sm rr.
struct Polar2 {
    float2 rr, cm, sm;
};

__device__ __forceinline__ Polar2 polar2(uint4 w) {
    // ---- radius ----
    const uint32_t ybA = __float_as_uint(__uint2float_rn((w.x & 0xFFFFFE00u) | 0x100u));
    const uint32_t ybB = __float_as_uint(__uint2float_rn((w.z & 0xFFFFFE00u) | 0x100u));
    const int32_t ixA = static_cast<int32_t>(ybA - 0x4F400000u);
    const int32_t ixB = static_cast<int32_t>(ybB - 0x4F400000u);
    const float2 f = make_float2(
        __uint_as_float((static_cast<uint32_t>(ixA) & 0x7FFFFFu) + 0x3F400000u),
        __uint_as_float((static_cast<uint32_t>(ixB) & 0x7FFFFFu) + 0x3F400000u));
    const float2 t = add2<kPackR>(f, splat(-1.0f));
    const float2 d = fma2<kPackR>(t, splat(0.25f), splat(0.5f));      // (2 + t) / 4
    const float2 q = mul2<kPackR>(t, make_float2(rcp_approx(d.x), rcp_approx(d.y)));  // 4t/(2+t)
    const float2 ww = mul2<kPackR>(q, q);
    float2 p = fma2<kPackR>(ww, splat(kLogR2), splat(kLogR1));
    p = fma2<kPackR>(ww, p, splat(kLogR0));
    const float2 lp = fma2<kPackR>(q, mul2<kPackR>(ww, p), q);          // 2 ln(1 + t)
    const float2 fe = make_float2(__int2float_rn(ixA >> 23), __int2float_rn(ixB >> 23));
    const float2 l_lo = fma2<kPackR>(fe, splat(-kTwoLn2Lo), lp);
    // e (2 ln 2)_hi is exact, so L is l_hi + l_lo rounded once
    const float2 L = fma2<kPackR>(fe, splat(-kTwoLn2Hi), l_lo);         // -(-2 ln u_a)
    Polar2 o;
    o.rr = make_float2(-sqrt_approx(-L.x), -sqrt_approx(-L.y));       // -r

    // ---- angle ----
    const int32_t waA = static_cast<int32_t>(((w.y << 2) & 0xFFFFFC00u) | 0x200u);
    const int32_t waB = static_cast<int32_t>(((w.w << 2) & 0xFFFFFC00u) | 0x200u);
    const float2 x = make_float2(__fmul_rn(fabsf(__int2float_rn(waA)), 0x1p-31f),
                                 __fmul_rn(fabsf(__int2float_rn(waB)), 0x1p-31f));
    const float2 y = mul2<kPackA>(x, x);
    float2 ps = fma2<kPackA>(y, splat(kSinS2), splat(kSinS1));
    ps = fma2<kPackA>(y, ps, splat(kSinS0));
    ps = fma2<kPackA>(y, ps, splat(kSinLo));
    const float2 S = fma2<kPackA>(x, splat(kSinHi), mul2<kPackA>(x, ps));
    float2 pc = fma2<kPackA>(y, splat(kCosC3), splat(kCosC2));
    pc = fma2<kPackA>(y, pc, splat(kCosC1));
    pc = fma2<kPackA>(y, pc, splat(kCosC0));
    const float2 C = fma2<kPackA>(y, pc, splat(1.0f));
    // octant bits o2 o1 o0 = word bits 31..29: |cos| and |sin| swap when o0 ^ o1;
    // cos < 0 when o1 ^ o2, sin < 0 when o2; one more flip for the negated radius
    const uint32_t tA = w.y ^ (w.y << 1), tB = w.w ^ (w.w << 1);
    const bool swA = (tA & 0x40000000u) != 0u, swB = (tB & 0x40000000u) != 0u;
    o.cm = make_float2(
        __uint_as_float(__float_as_uint(swA ? S.x : C.x) ^ (tA & 0x80000000u) ^ 0x80000000u),
        __uint_as_float(__float_as_uint(swB ? S.y : C.y) ^ (tB & 0x80000000u) ^ 0x80000000u));
    o.sm = make_float2(
        __uint_as_float(__float_as_uint(swA ? C.x : S.x) ^ (w.y & 0x80000000u) ^ 0x80000000u),
        __uint_as_float(__float_as_uint(swB ? C.y : S.y) ^ (w.w & 0x80000000u) ^ 0x80000000u));
    return o;
}

// even = (z of word pair A's even element, pair B's even element), odd likewise.
struct GaussPair {
    float2 even, odd;
};

__device__ __forceinline__ GaussPair box_muller2(uint4 w) {
    const Polar2 o = polar2(w);
    GaussPair g;
    g.even = mul2<kPackO>(o.cm, o.rr);
    g.odd = mul2<kPackO>(o.sm, o.rr);
    return g;
}

// The four Gaussians of block (b_lo, b_hi), elements 4b .. 4b + 3.
__device__ __forceinline__ float4 block_gaussians(const SeedConst& s, uint32_t b_lo, uint32_t b_hi) {
    const GaussPair g = box_muller2(philox_block(s, b_lo, b_hi));
    return make_float4(g.even.x, g.odd.x, g.even.y, g.odd.y);
}

}  // namespace jb

