// jb_kernels.cu -- sm_103a kernels of the seeded-perturbation hot path.
//
//   seeded_kernel<T, false>  PerturbParameters(theta, eps, s) (Algorithm 1,
//                            subroutine): theta_e <- round_T(theta_e + eps z_e),
//                            one fused multiply-add fma(s_e, eps r_e, theta_e).
//   seeded_kernel<T, true>   the step update (Section 2; Algorithm 1):
//                            theta_e <- round_T(theta_e + sum_k c_k z_e(s_k)),
//                            the K pairs regenerated in registers, so theta is
//                            read once and written once whatever K is.
//   general_update_kernel<T> the update read from one table and written to
//                            another, seeds in groups rounded to T after each
//                            (the backup-fused restore and the multi-step replay).
//   checksum_kernel<T>       the model checksum of ChecksumMatch (Algorithm 1).
//   debug kernels            raw Philox words, z by element, Box-Muller of given
//                            words (test hooks only).
//
// Design. Nothing here is a dense contraction, so there is no tensor-core
// work: the cost is one HBM read and write of theta (2 sizeof(T) bytes per
// element) against K Gaussians per element (a quarter Philox4x32-10 block and
// half a Box-Muller transform each). The grid is persistent (a multiple of the
// SM count times the resident CTAs per SM) and strides over spans of S warp
// tiles: a warp tile is 32 * V consecutive 16-byte vectors, lane l taking
// vectors l, l + 32, ..., so every load and store instruction of a warp covers
// 512 contiguous bytes (fully coalesced, 128-bit per thread). Each thread keeps
// V vectors in flight for instruction-level parallelism; the segment lookup
// (64-bit index arithmetic) is paid once per span, not once per tile.
// The K (seed, coefficient) pairs live in the kernel parameter space and are
// read with warp-uniform indices (constant-bank broadcast). Accumulation is a
// fixed-order fp32 FMA chain with no atomics: results are bitwise repeatable
// and independent of the grid and of how tensors are split.
#include <cuda_bf16.h>

#include <atomic>
#include <mutex>

#include "jb_internal.h"
#include "jb_rng.cuh"

namespace jb {
namespace {

#ifndef JB_V_F32
#define JB_V_F32 4
#endif
#ifndef JB_V_BF16
#define JB_V_BF16 2
#endif
#ifndef JB_MIN_CTAS_UPDATE  // 0: no occupancy hint to ptxas
#define JB_MIN_CTAS_UPDATE 0
#endif
#ifndef JB_MIN_CTAS_PERTURB
#define JB_MIN_CTAS_PERTURB 0
#endif

#ifndef JB_VP_F32
#define JB_VP_F32 4
#endif
#ifndef JB_VP_BF16
#define JB_VP_BF16 4
#endif
#ifndef JB_SU_F32  // warp tiles per span, update kernels
#define JB_SU_F32 4
#endif
#ifndef JB_SU_BF16
#define JB_SU_BF16 4
#endif
#ifndef JB_SG_F32  // warp tiles per span, general update kernel
#define JB_SG_F32 4
#endif
#ifndef JB_SG_BF16
#define JB_SG_BF16 4
#endif
#ifndef JB_SP_F32  // warp tiles per span, perturb kernel
#define JB_SP_F32 4
#endif
#ifndef JB_SP_BF16
#define JB_SP_BF16 4
#endif
#ifndef JB_PIPE_F32
#define JB_PIPE_F32 0
#endif
#ifndef JB_PIPE_BF16
#define JB_PIPE_BF16 1
#endif

// Per storage type: elements per 16-byte vector, vectors per thread per warp tile,
// warp tiles per span (the unit whose segment lookup is done once), and whether
// the update loop computes seed k + 1's Philox words while seed k is transformed
// (measured faster for bf16, slower for fp32 at these tile sizes).
template <typename T>
struct Traits;
template <>
struct Traits<float> {
    static constexpr int E = 4;
    static constexpr int V = JB_V_F32;
    static constexpr bool PIPE = JB_PIPE_F32;
    static constexpr int VP = JB_VP_F32;  // vectors per thread, perturb
    static constexpr int SU = JB_SU_F32;  // tiles per span, update
    static constexpr int SG = JB_SG_F32;  // tiles per span, general update
    static constexpr int SP = JB_SP_F32;  // tiles per span, perturb
};
template <>
struct Traits<__nv_bfloat16> {
    static constexpr int E = 8;
    static constexpr int V = JB_V_BF16;
    static constexpr bool PIPE = JB_PIPE_BF16;
    static constexpr int VP = JB_VP_BF16;
    static constexpr int SU = JB_SU_BF16;
    static constexpr int SG = JB_SG_BF16;
    static constexpr int SP = JB_SP_BF16;
};

__device__ __forceinline__ void load_vec(const float* p, float (&x)[4]) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(p));
    x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
}
__device__ __forceinline__ void store_vec(float* p, const float (&x)[4]) {
    __stcs(reinterpret_cast<float4*>(p), make_float4(x[0], x[1], x[2], x[3]));
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // nearest, ties to even
    return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ void load_vec(const __nv_bfloat16* p, float (&x)[8]) {
    const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p));
    x[0] = bf16_lo(v.x); x[1] = bf16_hi(v.x); x[2] = bf16_lo(v.y); x[3] = bf16_hi(v.y);
    x[4] = bf16_lo(v.z); x[5] = bf16_hi(v.z); x[6] = bf16_lo(v.w); x[7] = bf16_hi(v.w);
}
__device__ __forceinline__ void store_vec(__nv_bfloat16* p, const float (&x)[8]) {
    __stcs(reinterpret_cast<uint4*>(p), make_uint4(pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]),
                                                   pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7])));
}
__device__ __forceinline__ float load_one(const float* p) { return *p; }
__device__ __forceinline__ void store_one(float* p, float v) { *p = v; }
__device__ __forceinline__ float load_one(const __nv_bfloat16* p) {
    return __uint_as_float(static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(p)) << 16);
}
__device__ __forceinline__ void store_one(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

__device__ __forceinline__ Key seed_key(const SeedParam& s) {
    Key k;
    k.k0 = s.k0; k.k1 = s.k1; k.step = s.step; k.sample = s.sample;
    return k;
}


// Philox words of the B blocks of each of V vectors (blk[j] is a multiple of B, so
// adding b never carries into the high word).
template <int V, int B>
__device__ __forceinline__ void tile_words(const SeedConst& sc, const uint64_t (&blk)[V],
                                           uint4 (&w)[V][B]) {
#pragma unroll
    for (int j = 0; j < V; ++j)
#pragma unroll
        for (int b = 0; b < B; ++b)
            w[j][b] = philox_block(sc, static_cast<uint32_t>(blk[j]) + b,
                                   static_cast<uint32_t>(blk[j] >> 32));
}

// acc_even += c z_even, acc_odd += c z_odd for the Gaussians of one Philox block.
// The scale c is applied to the radius (rc = c r, rounded once) and each product
// c z is formed as one fused multiply-add of the signed cosine or sine with rc: one
// packed multiply fewer per block than scaling z = cos r after it is rounded.
__device__ __forceinline__ void accum_block(uint4 w, float2 c, float2& acc_even, float2& acc_odd) {
    const Polar2 o = polar2(w);
    const float2 rc = mul2<kPackO>(c, o.rr);
    acc_even = fma2<kPackO>(o.cm, rc, acc_even);
    acc_odd = fma2<kPackO>(o.sm, rc, acc_odd);
}

// acc += c z for the Gaussians of the words w; accumulators are packed per block as
// (elements 4b, 4b + 2) and (4b + 1, 4b + 3).
template <int V, int B>
__device__ __forceinline__ void tile_accumulate(const uint4 (&w)[V][B], float c,
                                                float2 (&acc)[V][B][2]) {
#pragma unroll
    for (int j = 0; j < V; ++j)
#pragma unroll
        for (int b = 0; b < B; ++b) accum_block(w[j][b], splat(c), acc[j][b][0], acc[j][b][1]);
}

template <typename T, bool UPDATE>
struct MinCtas {
    static constexpr int value = UPDATE ? JB_MIN_CTAS_UPDATE : JB_MIN_CTAS_PERTURB;
};

// One thread's share of a warp tile: V vectors of E elements, as fp32 values,
// with the segment, first Philox block and vector-path flag of each vector.
template <typename T, int V>
struct Tile {
    static constexpr int E = Traits<T>::E;
    float x[V][E];
    uint32_t seg[V];
    uint64_t blk[V];
    bool full[V];
};

__device__ __forceinline__ uint64_t dst_address(const SegParam& g) { return g.ptr & ~1ull; }
__device__ __forceinline__ uint64_t dst_address(const SegParamOut& g) { return g.dst; }

// Warp-uniform description of a warp tile that lies inside one segment with every
// vector full and on the 16-byte path (the common case): vector 32 j + lane of the
// tile is at base + (32 j + lane) * 16 bytes and starts at global window
// win0 + 32 j + lane. Every lane computes the same values, so branching on `fast`
// does not diverge; other tiles take the per-vector path of load_tile/store_tile.
struct TileFast {
    bool fast;
    uint32_t count;  // vectors in the tile
    uint64_t base;   // source address of the tile's first vector
    uint64_t dst;    // destination address of the tile's first vector
    uint64_t win0;   // global window (E-element group) of the first vector
};

template <int E, int V, int ES, typename P>
__device__ __forceinline__ TileFast tile_fast(const P& p, uint64_t wt, uint32_t& s) {
    const uint64_t v0 = wt * (32u * V);
    const uint64_t n_vec = p.n_vec;
    while (s + 1 < p.n_segs && p.segs[s + 1].vec0 <= v0) ++s;
    const auto& g = p.segs[s];
    const uint64_t seg_end = s + 1 < p.n_segs ? p.segs[s + 1].vec0 : n_vec;
    const uint64_t vend = v0 + 32u * V < n_vec ? v0 + 32u * V : n_vec;
    TileFast f;
    f.win0 = g.fo / E + (v0 - g.vec0);
    const int64_t i_first = static_cast<int64_t>(f.win0 * E) - static_cast<int64_t>(g.fo);
    const int64_t i_end = i_first + static_cast<int64_t>(vend - v0) * E;
    f.fast = vend <= seg_end && (g.ptr & 1ull) && i_first >= 0 && i_end <= static_cast<int64_t>(g.n);
    f.count = static_cast<uint32_t>(vend - v0);
    f.base = (g.ptr & ~1ull) + static_cast<uint64_t>(i_first) * ES;
    f.dst = dst_address(g) + static_cast<uint64_t>(i_first) * ES;
    return f;
}

// Loads tile wt. The segment cursor s only moves forward: a thread's vector
// indices grow from one call to the next.
template <typename T, int V, typename P>
__device__ __forceinline__ void load_tile(const P& p, uint64_t wt, uint32_t lane, uint32_t& s,
                                          Tile<T, V>& tl) {
    constexpr int E = Traits<T>::E;
    const uint64_t n_vec = p.n_vec;
    const uint32_t n_segs = p.n_segs;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const uint64_t vi = wt * (32u * V) + 32u * j + lane;
        const bool valid = vi < n_vec;
        if (valid)
            while (s + 1 < n_segs && p.segs[s + 1].vec0 <= vi) ++s;
        tl.seg[j] = s;
        const auto& g = p.segs[s];
        const uint64_t e0 = (g.fo / E + (vi - g.vec0)) * E;
        tl.blk[j] = e0 >> 2;
        const int64_t i0 = static_cast<int64_t>(e0) - static_cast<int64_t>(g.fo);
        const int64_t n = static_cast<int64_t>(g.n);
        const T* base = reinterpret_cast<const T*>(g.ptr & ~1ull);
        tl.full[j] = valid && (g.ptr & 1ull) && i0 >= 0 && i0 + E <= n;
        if (tl.full[j]) {
            load_vec(base + i0, tl.x[j]);
        } else {
#pragma unroll
            for (int t = 0; t < E; ++t) {
                const int64_t i = i0 + t;
                tl.x[j][t] = (valid && i >= 0 && i < n) ? load_one(base + i) : 0.0f;
            }
        }
    }
}

template <typename T, int V, bool TO_DST = false, typename P>
__device__ __forceinline__ void store_tile(const P& p, uint64_t wt, uint32_t lane,
                                           const Tile<T, V>& tl) {
    constexpr int E = Traits<T>::E;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const uint64_t vi = wt * (32u * V) + 32u * j + lane;
        if (vi >= p.n_vec) continue;
        const auto& g = p.segs[tl.seg[j]];
        T* base;
        if constexpr (TO_DST) base = reinterpret_cast<T*>(g.dst);
        else base = reinterpret_cast<T*>(g.ptr & ~1ull);
        const int64_t i0 = static_cast<int64_t>(tl.blk[j] << 2) - static_cast<int64_t>(g.fo);
        if (tl.full[j]) {
            store_vec(base + i0, tl.x[j]);
        } else {
            const int64_t n = static_cast<int64_t>(g.n);
#pragma unroll
            for (int t = 0; t < E; ++t) {
                const int64_t i = i0 + t;
                if (i >= 0 && i < n) store_one(base + i, tl.x[j][t]);
            }
        }
    }
}

// Runs op on each of this warp's tiles and stores the result (to the destination
// table when TO_DST, and then also back to the source when also_src). The warp
// takes spans of S consecutive warp tiles, strided by the number of warps in the
// grid. The segment lookup and fast-path test are done once per span: when the
// whole span lies inside one aligned segment, its tiles follow one another at
// fixed byte strides; otherwise each tile takes the per-vector path. Which warp
// handles a tile never changes a result: every element's value depends only on
// its own stored value, its global index and the seeds.
template <typename T, int V, int S, bool TO_DST, typename P, typename Op>
__device__ __forceinline__ void visit_tiles(const P& p, bool also_src, Op&& op) {
    constexpr int E = Traits<T>::E;
    constexpr uint32_t kTileVec = 32u * V;
    const uint32_t lane = threadIdx.x & 31u;
    const uint64_t warp = (static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const uint64_t n_warps = (static_cast<uint64_t>(gridDim.x) * kThreads) >> 5;
    const uint64_t n_vec = p.n_vec;
    uint32_t s = 0;  // segment cursor; only moves forward
    for (uint64_t ws = warp; ws * (kTileVec * S) < n_vec; ws += n_warps) {
        const TileFast fs = tile_fast<E, V * S, sizeof(T)>(p, ws, s);
        if (fs.fast) {
            // per-thread addresses and Philox blocks of the tile's vectors, advanced
            // by one tile's stride per tile instead of recomputed from the tile base
            constexpr uint64_t kStep = 16ull * kTileVec;
            uint64_t sp[V], dp[V], bk[V];
#pragma unroll
            for (int j = 0; j < V; ++j) {
                const uint64_t off = 16ull * (32u * j + lane);
                sp[j] = fs.base + off;
                dp[j] = fs.dst + off;
                bk[j] = (fs.win0 + 32u * j + lane) * (E / 4);
            }
#pragma unroll 1
            for (uint32_t done = 0; done < fs.count; done += kTileVec) {
                const uint32_t cnt = fs.count - done < kTileVec ? fs.count - done : kTileVec;
                Tile<T, V> tl;
#pragma unroll
                for (int j = 0; j < V; ++j) {
                    tl.blk[j] = bk[j];
                    tl.full[j] = 32u * j + lane < cnt;
                    tl.seg[j] = 0;
                    if (tl.full[j]) {
                        load_vec(reinterpret_cast<const T*>(sp[j]), tl.x[j]);
                    } else {
#pragma unroll
                        for (int t = 0; t < E; ++t) tl.x[j][t] = 0.0f;
                    }
                }
                op(tl);
#pragma unroll
                for (int j = 0; j < V; ++j) {
                    if (!tl.full[j]) continue;
                    store_vec(reinterpret_cast<T*>(TO_DST ? dp[j] : sp[j]), tl.x[j]);
                    if (TO_DST && also_src) store_vec(reinterpret_cast<T*>(sp[j]), tl.x[j]);
                }
#pragma unroll
                for (int j = 0; j < V; ++j) {
                    sp[j] += kStep;
                    dp[j] += kStep;
                    bk[j] += kTileVec * (E / 4);
                }
            }
        } else {
#pragma unroll 1
            for (int u = 0; u < S; ++u) {
                const uint64_t wt = ws * S + u;
                if (wt * kTileVec >= n_vec) break;
                Tile<T, V> tl;
                load_tile<T, V>(p, wt, lane, s, tl);
                op(tl);
                store_tile<T, V, TO_DST>(p, wt, lane, tl);
                if (TO_DST && also_src) store_tile<T, V, false>(p, wt, lane, tl);
            }
        }
    }
}

// acc = sum_{k in [kb, ke)} c_k z_k for the tile, in fp32, in seed order (ke > kb).
// SINGLE_PIPE: a range of one seed computes the Philox words of vector j + 1 while
// vector j is transformed (measured faster in the general update kernel, whose
// replay groups are often one seed, and slower in the in-place one).
template <typename T, int V, bool SINGLE_PIPE = false, typename P>
__device__ __forceinline__ void accumulate_range(const P& p, const uint64_t (&blk)[V], uint32_t kb,
                                                 uint32_t ke, float2 (&acc)[V][Traits<T>::E / 4][2]) {
    constexpr int B = Traits<T>::E / 4;  // Philox blocks per vector
#pragma unroll
    for (int j = 0; j < V; ++j)
#pragma unroll
        for (int b = 0; b < B; ++b) acc[j][b][0] = acc[j][b][1] = make_float2(0.0f, 0.0f);
    if constexpr (SINGLE_PIPE) {
        if (ke - kb == 1) {
            const SeedConst sc = seed_const(seed_key(p.seeds[kb]));
            const float c = p.seeds[kb].coef;
            uint4 wc[B], wn[B];
#pragma unroll
            for (int b = 0; b < B; ++b)
                wc[b] = philox_block(sc, static_cast<uint32_t>(blk[0]) + b, static_cast<uint32_t>(blk[0] >> 32));
#pragma unroll
            for (int j = 0; j < V; ++j) {
                if (j + 1 < V) {
#pragma unroll
                    for (int b = 0; b < B; ++b)
                        wn[b] = philox_block(sc, static_cast<uint32_t>(blk[j + 1]) + b,
                                             static_cast<uint32_t>(blk[j + 1] >> 32));
                }
#pragma unroll
                for (int b = 0; b < B; ++b) accum_block(wc[b], splat(c), acc[j][b][0], acc[j][b][1]);
                if (j + 1 < V) {
#pragma unroll
                    for (int b = 0; b < B; ++b) wc[b] = wn[b];
                }
            }
            return;
        }
    }
    if constexpr (Traits<T>::PIPE) {
        // Philox words of seed k + 1 are computed while seed k is transformed and
        // accumulated: the integer-multiply work and the fp32 work are independent
        // and interleave in one instruction stream. The last seed is peeled.
        uint4 w[V][B];
        tile_words<V, B>(seed_const(seed_key(p.seeds[kb])), blk, w);
        // per block: the next seed's Philox words, then this seed's transform
        // Philox round 1's product of the block counter is the same for every seed
        BlockCtr bc[V][B];
#pragma unroll
        for (int j = 0; j < V; ++j)
#pragma unroll
            for (int b = 0; b < B; ++b)
                bc[j][b] = block_ctr(static_cast<uint32_t>(blk[j]) + b, static_cast<uint32_t>(blk[j] >> 32));
        for (uint32_t k = kb; k + 1 < ke; ++k) {
            const SeedConst sn = seed_const(seed_key(p.seeds[k + 1]));
            const float2 c = splat(p.seeds[k].coef);
#pragma unroll
            for (int j = 0; j < V; ++j)
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const uint4 wn = philox_block(sn, bc[j][b]);
                    accum_block(w[j][b], c, acc[j][b][0], acc[j][b][1]);
                    w[j][b] = wn;
                }
        }
        tile_accumulate<V, B>(w, p.seeds[ke - 1].coef, acc);
    } else {
        for (uint32_t k = kb; k < ke; ++k) {
            uint4 w[V][B];
            tile_words<V, B>(seed_const(seed_key(p.seeds[k])), blk, w);
            tile_accumulate<V, B>(w, p.seeds[k].coef, acc);
        }
    }
}

// x += acc with one fp32 rounding; ROUND_T also rounds the sum to the storage type
// (between the steps of a replay, where the next step reads the stored value).
template <typename T, int V, bool ROUND_T>
__device__ __forceinline__ void add_acc(Tile<T, V>& tl, const float2 (&acc)[V][Traits<T>::E / 4][2]) {
    constexpr int B = Traits<T>::E / 4;
#pragma unroll
    for (int j = 0; j < V; ++j)
#pragma unroll
        for (int b = 0; b < B; ++b) {
            float v0 = __fadd_rn(tl.x[j][4 * b + 0], acc[j][b][0].x);
            float v2 = __fadd_rn(tl.x[j][4 * b + 2], acc[j][b][0].y);
            float v1 = __fadd_rn(tl.x[j][4 * b + 1], acc[j][b][1].x);
            float v3 = __fadd_rn(tl.x[j][4 * b + 3], acc[j][b][1].y);
            if constexpr (ROUND_T && sizeof(T) == 2) {
                v0 = __bfloat162float(__float2bfloat16_rn(v0));
                v1 = __bfloat162float(__float2bfloat16_rn(v1));
                v2 = __bfloat162float(__float2bfloat16_rn(v2));
                v3 = __bfloat162float(__float2bfloat16_rn(v3));
            }
            tl.x[j][4 * b + 0] = v0;
            tl.x[j][4 * b + 1] = v1;
            tl.x[j][4 * b + 2] = v2;
            tl.x[j][4 * b + 3] = v3;
        }
}

// theta += sum_k c_k z_k over the tile, accumulated in fp32 in seed order.
template <typename T, int V, typename P>
__device__ __forceinline__ void update_tile(const P& p, Tile<T, V>& tl) {
    float2 acc[V][Traits<T>::E / 4][2];
    accumulate_range<T, V>(p, tl.blk, 0, p.n_seeds, acc);
    add_acc<T, V, false>(tl, acc);
}

// One seed over the tile: ADD = false is the perturbation theta <- fma(., ., theta)
// (one rounding of theta + eps z); ADD = true is a one-pair update, theta <- theta +
// (c z rounded to fp32), the same arithmetic as update_tile with K = 1. The Philox
// words of vector j + 1 are computed while vector j is transformed, so the
// integer-multiply and fp32 work of neighbouring vectors interleave (as the update
// does across seeds).
template <typename T, int V, bool ADD, typename P>
__device__ __forceinline__ void one_seed_tile(const P& p, Tile<T, V>& tl) {
    constexpr int B = Traits<T>::E / 4;
    const SeedConst sc = seed_const(seed_key(p.seeds[0]));
    const float2 c = splat(p.seeds[0].coef);
    uint4 wc[B], wn[B];
#pragma unroll
    for (int b = 0; b < B; ++b)
        wc[b] = philox_block(sc, static_cast<uint32_t>(tl.blk[0]) + b, static_cast<uint32_t>(tl.blk[0] >> 32));
#pragma unroll
    for (int j = 0; j < V; ++j) {
        if (j + 1 < V) {
#pragma unroll
            for (int b = 0; b < B; ++b)
                wn[b] = philox_block(sc, static_cast<uint32_t>(tl.blk[j + 1]) + b,
                                     static_cast<uint32_t>(tl.blk[j + 1] >> 32));
        }
#pragma unroll
        for (int b = 0; b < B; ++b) {
            float* x = &tl.x[j][4 * b];
            if constexpr (ADD) {
                float2 ev = make_float2(0.0f, 0.0f), od = make_float2(0.0f, 0.0f);
                accum_block(wc[b], c, ev, od);
                x[0] = __fadd_rn(x[0], ev.x);
                x[2] = __fadd_rn(x[2], ev.y);
                x[1] = __fadd_rn(x[1], od.x);
                x[3] = __fadd_rn(x[3], od.y);
            } else {
                float2 ev = make_float2(x[0], x[2]), od = make_float2(x[1], x[3]);
                accum_block(wc[b], c, ev, od);
                x[0] = ev.x;
                x[2] = ev.y;
                x[1] = od.x;
                x[3] = od.y;
            }
        }
        if (j + 1 < V) {
#pragma unroll
            for (int b = 0; b < B; ++b) wc[b] = wn[b];
        }
    }
}

template <typename T, bool UPDATE, typename P>
__global__ void
#if JB_MIN_CTAS_UPDATE || JB_MIN_CTAS_PERTURB
__launch_bounds__(kThreads, (MinCtas<T, UPDATE>::value > 0 ? MinCtas<T, UPDATE>::value : 1))
#else
__launch_bounds__(kThreads)
#endif
    seeded_kernel(const __grid_constant__ P p) {
    constexpr int V = UPDATE ? Traits<T>::V : Traits<T>::VP;
    constexpr int S = UPDATE ? Traits<T>::SU : Traits<T>::SP;
    visit_tiles<T, V, S, false>(p, false, [&](Tile<T, V>& tl) {
        if constexpr (UPDATE) update_tile<T, V>(p, tl);
        else one_seed_tile<T, V, false>(p, tl);
    });
}

// A one-pair update (K = 1, one group) in the perturbation's tile shape: in place
// (TO_DST = false) or from the source table to the destination (and back to the
// source when write_src).
template <typename T, bool TO_DST, typename P>
__global__ void __launch_bounds__(kThreads) one_pair_kernel(const __grid_constant__ P p) {
    constexpr int V = Traits<T>::VP;
    bool also_src = false;
    if constexpr (TO_DST) also_src = p.write_src != 0;
    visit_tiles<T, V, Traits<T>::SP, TO_DST>(p, also_src, [&](Tile<T, V>& tl) {
        one_seed_tile<T, V, true>(p, tl);
    });
}

// The generalised update: source -> destination (optionally also back to the
// source), seeds applied in groups with a rounding to the storage type after each
// group, exactly as successive in-place updates would round.
template <typename T>
__global__ void __launch_bounds__(kThreads) general_update_kernel(const __grid_constant__ GeneralParams p) {
    constexpr int V = Traits<T>::V;
    visit_tiles<T, V, Traits<T>::SG, true>(p, p.write_src != 0, [&](Tile<T, V>& tl) {
        uint32_t kb = 0;
        for (uint32_t g = 0; g < p.n_groups; ++g) {
            const uint32_t ke = p.group_end[g];  // > kb: the host drops empty groups
            float2 acc[V][Traits<T>::E / 4][2];
            accumulate_range<T, V, true>(p, tl.blk, kb, ke, acc);
            // the store rounds the last group's sum to T; rounding twice to the
            // nearest gives the same bits, so only earlier groups round here
            if (g + 1 < p.n_groups) add_acc<T, V, true>(tl, acc);
            else add_acc<T, V, false>(tl, acc);
            kb = ke;
        }
    });
}

// Model checksum (ChecksumMatch, Algorithm 1): the sum mod 2^64, over 16-byte
// windows of the global element space, of four Philox rounds of the window's
// storage words (elements outside the segment read as 0) keyed by the window
// index; per window (x1:x0) + (x3:x2). Integer addition is order-free, so one
// atomic add per CTA gives the same bits for any grid. Bound by HBM: one read
// of theta, one wide multiply pair per window and round.
constexpr uint32_t kSumKey0 = 0x6A09E667u, kSumKey1 = 0xF3BCC908u;
constexpr int kSumRounds = 4;
#ifndef JB_SUM_V
#define JB_SUM_V 8
#endif
constexpr int kSumV = JB_SUM_V;  // 16-byte loads in flight per thread
#ifndef JB_SUM_S
#define JB_SUM_S 4
#endif
constexpr int kSumS = JB_SUM_S;  // warp tiles per span

__device__ __forceinline__ uint64_t window_hash(uint64_t win, uint4 w) {
    uint32_t x0 = w.x, x1 = w.y, x2 = w.z, x3 = w.w;
    uint32_t k0 = static_cast<uint32_t>(win) ^ kSumKey0;
    uint32_t k1 = static_cast<uint32_t>(win >> 32) ^ kSumKey1;
#pragma unroll
    for (int r = 0; r < kSumRounds; ++r) {
        if (r > 0) {
            k0 += kPhiloxW0;
            k1 += kPhiloxW1;
        }
        philox_round(x0, x1, x2, x3, k0, k1);
    }
    return ((static_cast<uint64_t>(x1) << 32) | x0) + ((static_cast<uint64_t>(x3) << 32) | x2);
}

__device__ __forceinline__ uint32_t raw_bits(const float* p) { return __float_as_uint(*p); }
__device__ __forceinline__ uint32_t raw_bits(const __nv_bfloat16* p) {
    return *reinterpret_cast<const uint16_t*>(p);
}

// Checksum terms of warp tile wt on the per-vector path (tiles that cross a
// segment boundary or lie in a segment off the 16-byte grid): windows are read
// element by element where they are partial, with elements outside the segment
// taken as zero bits.
template <typename T, int V>
__device__ __forceinline__ uint64_t sum_tile_general(const PerturbParams& p, uint64_t wt, uint32_t lane,
                                                     uint32_t& s) {
    constexpr int E = Traits<T>::E;
    constexpr int BITS = 8 * static_cast<int>(sizeof(T));
    const uint64_t n_vec = p.n_vec;
    const uint32_t n_segs = p.n_segs;
    uint64_t sum = 0;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const uint64_t vi = wt * (32u * V) + 32u * j + lane;
        const bool valid = vi < n_vec;
        if (valid)
            while (s + 1 < n_segs && p.segs[s + 1].vec0 <= vi) ++s;
        const SegParam& g = p.segs[s];
        const uint64_t win = g.fo / E + (vi - g.vec0);
        const int64_t i0 = static_cast<int64_t>(win * E) - static_cast<int64_t>(g.fo);
        const int64_t n = static_cast<int64_t>(g.n);
        const T* base = reinterpret_cast<const T*>(g.ptr & ~1ull);
        uint4 w;
        if (valid && (g.ptr & 1ull) && i0 >= 0 && i0 + E <= n) {
            w = __ldcs(reinterpret_cast<const uint4*>(base + i0));
        } else {
            uint32_t ww[4] = {0u, 0u, 0u, 0u};
#pragma unroll
            for (int t = 0; t < E; ++t) {
                const int64_t i = i0 + t;
                if (valid && i >= 0 && i < n) ww[t * BITS / 32] |= raw_bits(base + i) << ((t * BITS) % 32);
            }
            w = make_uint4(ww[0], ww[1], ww[2], ww[3]);
        }
        if (valid) sum += window_hash(win, w);
    }
    return sum;
}

template <typename T>
__global__ void __launch_bounds__(kThreads) checksum_kernel(const __grid_constant__ PerturbParams p,
                                                           unsigned long long* out) {
    constexpr int E = Traits<T>::E;
    constexpr int V = kSumV;
    const uint32_t lane = threadIdx.x & 31u;
    const uint64_t warp = (static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const uint64_t n_warps = (static_cast<uint64_t>(gridDim.x) * kThreads) >> 5;
    const uint64_t n_vec = p.n_vec;
    constexpr int S = kSumS;
    constexpr uint32_t kTileVec = 32u * V;
    uint32_t s = 0;
    uint64_t sum = 0;
    for (uint64_t ws = warp; ws * (kTileVec * S) < n_vec; ws += n_warps) {
        const TileFast fs = tile_fast<E, V * S, sizeof(T)>(p, ws, s);
        if (fs.fast) {
#pragma unroll 1
            for (uint32_t done = 0; done < fs.count; done += kTileVec) {
                const uint64_t base = fs.base + 16ull * done;
                uint4 w[V];
                uint64_t win[V];
                bool valid[V];
#pragma unroll
                for (int j = 0; j < V; ++j) {
                    const uint32_t v = 32u * j + lane;
                    valid[j] = done + v < fs.count;
                    win[j] = fs.win0 + done + v;
                    w[j] = valid[j] ? __ldcs(reinterpret_cast<const uint4*>(base + 16ull * v))
                                    : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int j = 0; j < V; ++j)
                    if (valid[j]) sum += window_hash(win[j], w[j]);
            }
            continue;
        }
#pragma unroll 1
        for (int u = 0; u < S; ++u) {
            const uint64_t wt = ws * S + u;
            if (wt * kTileVec >= n_vec) break;
            sum += sum_tile_general<T, V>(p, wt, lane, s);
        }
    }
    // CTA reduction; every thread reaches the barrier
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) sum += __shfl_down_sync(0xFFFFFFFFu, sum, d);
    __shared__ uint64_t part[kThreads / 32];
    if (lane == 0) part[threadIdx.x >> 5] = sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint64_t t = 0;
#pragma unroll
        for (int i = 0; i < kThreads / 32; ++i) t += part[i];
        atomicAdd(out, static_cast<unsigned long long>(t));
    }
}

__global__ void debug_philox_kernel(SeedParam sp, uint64_t first, uint64_t n, uint32_t* out) {
    const uint64_t i = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const uint64_t b = first + i;
    const uint4 w = philox_block(seed_const(seed_key(sp)), static_cast<uint32_t>(b),
                                 static_cast<uint32_t>(b >> 32));
    reinterpret_cast<uint4*>(out)[i] = w;
}

// The Philox words of blocks [first, first + n) folded by XOR into *out: the
// generator alone, with the hot path's block function, on a persistent grid (each
// thread keeps kFoldIlp blocks in flight). XOR is order-free, so the result does
// not depend on the grid.
constexpr int kFoldIlp = 4;

__global__ void __launch_bounds__(kThreads) debug_philox_fold_kernel(SeedParam sp, uint64_t first,
                                                                    uint64_t n, uint32_t* out) {
    const SeedConst sc = seed_const(seed_key(sp));
    const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kThreads;
    uint32_t acc = 0;
    for (uint64_t i = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x; i < n;
         i += kFoldIlp * stride) {
#pragma unroll
        for (int u = 0; u < kFoldIlp; ++u) {
            const uint64_t j = i + u * stride;
            const uint64_t b = first + j;
            const uint4 w = philox_block(sc, static_cast<uint32_t>(b), static_cast<uint32_t>(b >> 32));
            if (j < n) acc ^= w.x ^ w.y ^ w.z ^ w.w;
        }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) acc ^= __shfl_xor_sync(0xFFFFFFFFu, acc, d);
    if ((threadIdx.x & 31u) == 0) atomicXor(out, acc);
}

__global__ void debug_gaussian_kernel(SeedParam sp, uint64_t first, uint64_t n, float* out) {
    const uint64_t i = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const uint64_t e = first + i;
    const uint64_t b = e >> 2;
    const float4 z = block_gaussians(seed_const(seed_key(sp)), static_cast<uint32_t>(b),
                                     static_cast<uint32_t>(b >> 32));
    const unsigned w = static_cast<unsigned>(e & 3u);
    out[i] = w == 0 ? z.x : (w == 1 ? z.y : (w == 2 ? z.z : z.w));
}

__global__ void debug_box_muller_kernel(const uint32_t* words, uint64_t n, float* out) {
    // the transform runs on two word pairs at once, as in the kernels above
    const uint64_t i = 2 * (static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x);
    if (i >= n) return;
    const uint64_t i1 = i + 1 < n ? i + 1 : i;
    const GaussPair g = box_muller2(make_uint4(words[2 * i], words[2 * i + 1], words[2 * i1],
                                               words[2 * i1 + 1]));
    out[2 * i] = g.even.x;
    out[2 * i + 1] = g.odd.x;
    if (i + 1 < n) {
        out[2 * i + 2] = g.even.y;
        out[2 * i + 3] = g.odd.y;
    }
}

// Persistent grid: SM count x resident CTAs per SM, cached per device and kernel.
constexpr int kMaxDevices = 64;
constexpr int kKernels = 13;
std::atomic<int> g_grid_cache[kMaxDevices][kKernels];

template <typename K>
cudaError_t persistent_grid(K kernel, int slot, int* grid) {
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < kMaxDevices) {
        const int cached = g_grid_cache[dev][slot].load(std::memory_order_relaxed);
        if (cached > 0) {
            *grid = cached;
            return cudaSuccess;
        }
    }
    int sms = 0, per_sm = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, 0);
    if (err != cudaSuccess) return err;
    *grid = sms * (per_sm > 0 ? per_sm : 1);
    if (dev < kMaxDevices) g_grid_cache[dev][slot].store(*grid, std::memory_order_relaxed);
    return cudaSuccess;
}

template <typename T, bool UPDATE, typename P>
cudaError_t launch_seeded(const P& p, int slot, int grid_ctas, cudaStream_t stream) {
    if (p.n_vec == 0) return cudaSuccess;
    auto kernel = seeded_kernel<T, UPDATE, P>;
    int grid = grid_ctas;
    if (grid <= 0) {
        cudaError_t err = persistent_grid(kernel, slot, &grid);
        if (err != cudaSuccess) return err;
        constexpr uint64_t vec_per_cta =
            32ull * (UPDATE ? Traits<T>::V * Traits<T>::SU : Traits<T>::VP * Traits<T>::SP) * (kThreads / 32);
        const uint64_t needed = (p.n_vec + vec_per_cta - 1) / vec_per_cta;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    kernel<<<grid, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

template <typename T, bool TO_DST, typename P>
cudaError_t launch_one_pair_t(const P& p, int slot, int grid_ctas, cudaStream_t stream) {
    if (p.n_vec == 0) return cudaSuccess;
    auto kernel = one_pair_kernel<T, TO_DST, P>;
    int grid = grid_ctas;
    if (grid <= 0) {
        cudaError_t err = persistent_grid(kernel, slot, &grid);
        if (err != cudaSuccess) return err;
        constexpr uint64_t vec_per_cta = 32ull * Traits<T>::VP * Traits<T>::SP * (kThreads / 32);
        const uint64_t needed = (p.n_vec + vec_per_cta - 1) / vec_per_cta;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    kernel<<<grid, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_update(const UpdateParams& p, int dtype, int grid_ctas, cudaStream_t s) {
    // one pair: the perturbation's tile shape (4 vectors per thread, the next
    // vector's Philox words during the current transform) is faster for one seed
    if (p.n_seeds == 1) {
        if (dtype == kF32) return launch_one_pair_t<float, false>(p, 9, grid_ctas, s);
        return launch_one_pair_t<__nv_bfloat16, false>(p, 10, grid_ctas, s);
    }
    if (dtype == kF32) return launch_seeded<float, true>(p, 0, grid_ctas, s);
    return launch_seeded<__nv_bfloat16, true>(p, 1, grid_ctas, s);
}

template <typename T>
cudaError_t launch_general_t(const GeneralParams& p, int slot, int grid_ctas, cudaStream_t stream) {
    if (p.n_vec == 0) return cudaSuccess;
    auto kernel = general_update_kernel<T>;
    int grid = grid_ctas;
    if (grid <= 0) {
        cudaError_t err = persistent_grid(kernel, slot, &grid);
        if (err != cudaSuccess) return err;
        constexpr uint64_t vec_per_cta = 32ull * Traits<T>::V * Traits<T>::SG * (kThreads / 32);
        const uint64_t needed = (p.n_vec + vec_per_cta - 1) / vec_per_cta;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    kernel<<<grid, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_general(const GeneralParams& p, int dtype, int grid_ctas, cudaStream_t s) {
    if (p.n_groups == 1 && p.n_seeds == 1) {
        if (dtype == kF32) return launch_one_pair_t<float, true>(p, 11, grid_ctas, s);
        return launch_one_pair_t<__nv_bfloat16, true>(p, 12, grid_ctas, s);
    }
    if (dtype == kF32) return launch_general_t<float>(p, 4, grid_ctas, s);
    return launch_general_t<__nv_bfloat16>(p, 5, grid_ctas, s);
}

template <typename T>
cudaError_t launch_checksum_t(const PerturbParams& p, unsigned long long* out, int slot,
                              int grid_ctas, cudaStream_t stream) {
    if (p.n_vec == 0) return cudaSuccess;
    auto kernel = checksum_kernel<T>;
    int grid = grid_ctas;
    if (grid <= 0) {
        cudaError_t err = persistent_grid(kernel, slot, &grid);
        if (err != cudaSuccess) return err;
        constexpr uint64_t vec_per_cta = 32ull * kSumV * kSumS * (kThreads / 32);
        const uint64_t needed = (p.n_vec + vec_per_cta - 1) / vec_per_cta;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    kernel<<<grid, kThreads, 0, stream>>>(p, out);
    return cudaGetLastError();
}

cudaError_t launch_checksum(const PerturbParams& p, int dtype, unsigned long long* out,
                            int grid_ctas, cudaStream_t s) {
    if (dtype == kF32) return launch_checksum_t<float>(p, out, 6, grid_ctas, s);
    return launch_checksum_t<__nv_bfloat16>(p, out, 7, grid_ctas, s);
}

cudaError_t launch_perturb(const PerturbParams& p, int dtype, int grid_ctas, cudaStream_t s) {
    if (dtype == kF32) return launch_seeded<float, false>(p, 2, grid_ctas, s);
    return launch_seeded<__nv_bfloat16, false>(p, 3, grid_ctas, s);
}

static unsigned blocks_for(uint64_t n) { return static_cast<unsigned>((n + 255) / 256); }

cudaError_t launch_debug_philox(SeedParam seed, uint64_t first, uint64_t n, uint32_t* out,
                                cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    debug_philox_kernel<<<blocks_for(n), 256, 0, s>>>(seed, first, n, out);
    return cudaGetLastError();
}

cudaError_t launch_debug_philox_fold(SeedParam seed, uint64_t first, uint64_t n, uint32_t* out,
                                     cudaStream_t s) {
    cudaError_t err = cudaMemsetAsync(out, 0, sizeof(uint32_t), s);
    if (err != cudaSuccess || n == 0) return err;
    int grid = 0;
    err = persistent_grid(debug_philox_fold_kernel, 8, &grid);
    if (err != cudaSuccess) return err;
    const uint64_t needed = (n + kThreads - 1) / kThreads;
    if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    debug_philox_fold_kernel<<<grid, kThreads, 0, s>>>(seed, first, n, out);
    return cudaGetLastError();
}

cudaError_t launch_debug_gaussian(SeedParam seed, uint64_t first, uint64_t n, float* out,
                                  cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    debug_gaussian_kernel<<<blocks_for(n), 256, 0, s>>>(seed, first, n, out);
    return cudaGetLastError();
}

cudaError_t launch_debug_box_muller(const uint32_t* words, uint64_t n, float* out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    debug_box_muller_kernel<<<blocks_for((n + 1) / 2), 256, 0, s>>>(words, n, out);
    return cudaGetLastError();
}

}  // namespace jb
