// jb_kernels.cu -- sm_103a kernels of the seeded-perturbation hot path.
//
//   seeded_kernel<T, false>  PerturbParameters(theta, eps, s) (Algorithm 1,
//                            subroutine): theta_e <- round_T(fma(eps, z_e, theta_e)).
//   seeded_kernel<T, true>   the step update (Section 2; Algorithm 1):
//                            theta_e <- round_T(theta_e + sum_k c_k z_e(s_k)),
//                            the K pairs regenerated in registers, so theta is
//                            read once and written once whatever K is.
//   debug kernels            raw Philox words, z by element, Box-Muller of given
//                            words (test hooks only).
//
// Design. Nothing here is a dense contraction, so there is no tensor-core
// work: the cost is one HBM read and write of theta (2 sizeof(T) bytes per
// element) against K Gaussians per element (a quarter Philox4x32-10 block and
// half a Box-Muller transform each). The grid is persistent (a multiple of the
// SM count times the resident CTAs per SM) and strides over warp tiles: a warp
// tile is 32 * V consecutive 16-byte vectors, lane l taking vectors l, l + 32,
// ..., so every load and store instruction of a warp covers 512 contiguous
// bytes (fully coalesced, 128-bit per thread). Each thread keeps V vectors
// (16 elements, 4 Philox blocks) in flight for instruction-level parallelism.
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

#ifndef JB_PIPE_F32
#define JB_PIPE_F32 0
#endif
#ifndef JB_PIPE_BF16
#define JB_PIPE_BF16 1
#endif

// Per storage type: elements per 16-byte vector, vectors per thread per warp tile,
// and whether the update loop computes seed k + 1's Philox words while seed k is
// transformed (measured faster for bf16, slower for fp32 at these tile sizes).
template <typename T>
struct Traits;
template <>
struct Traits<float> {
    static constexpr int E = 4;
    static constexpr int V = JB_V_F32;
    static constexpr bool PIPE = JB_PIPE_F32;
};
template <>
struct Traits<__nv_bfloat16> {
    static constexpr int E = 8;
    static constexpr int V = JB_V_BF16;
    static constexpr bool PIPE = JB_PIPE_BF16;
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

// acc += c z for the Gaussians of the words w; accumulators are packed per block as
// (elements 4b, 4b + 2) and (4b + 1, 4b + 3).
template <int V, int B>
__device__ __forceinline__ void tile_accumulate(const uint4 (&w)[V][B], float c,
                                                float2 (&acc)[V][B][2]) {
#pragma unroll
    for (int j = 0; j < V; ++j)
#pragma unroll
        for (int b = 0; b < B; ++b) {
            const GaussPair g = box_muller2(w[j][b]);
            acc[j][b][0] = fma2<kPackO>(splat(c), g.even, acc[j][b][0]);
            acc[j][b][1] = fma2<kPackO>(splat(c), g.odd, acc[j][b][1]);
        }
}

template <typename T, bool UPDATE>
struct MinCtas {
    static constexpr int value = UPDATE ? JB_MIN_CTAS_UPDATE : JB_MIN_CTAS_PERTURB;
};

template <typename T, bool UPDATE, typename P>
__global__ void
#if JB_MIN_CTAS_UPDATE || JB_MIN_CTAS_PERTURB
__launch_bounds__(kThreads, (MinCtas<T, UPDATE>::value > 0 ? MinCtas<T, UPDATE>::value : 1))
#else
__launch_bounds__(kThreads)
#endif
    seeded_kernel(const __grid_constant__ P p) {
    constexpr int E = Traits<T>::E;
    constexpr int V = Traits<T>::V;
    constexpr int B = E / 4;  // Philox blocks per vector
    const uint32_t lane = threadIdx.x & 31u;
    const uint64_t warp = (static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const uint64_t n_warps = (static_cast<uint64_t>(gridDim.x) * kThreads) >> 5;
    const uint64_t n_vec = p.n_vec;
    const uint32_t n_segs = p.n_segs;
    uint32_t s = 0;  // segment cursor: vector indices only grow within a thread

    for (uint64_t wt = warp; wt * (32u * V) < n_vec; wt += n_warps) {
        float x[V][E];
        uint32_t seg[V];
        uint64_t blk[V];
        bool full[V];
#pragma unroll
        for (int j = 0; j < V; ++j) {
            const uint64_t vi = wt * (32u * V) + 32u * j + lane;
            const bool valid = vi < n_vec;
            if (valid)
                while (s + 1 < n_segs && p.segs[s + 1].vec0 <= vi) ++s;
            seg[j] = s;
            const SegParam& g = p.segs[s];
            const uint64_t e0 = (g.fo / E + (vi - g.vec0)) * E;
            blk[j] = e0 >> 2;
            const int64_t i0 = static_cast<int64_t>(e0) - static_cast<int64_t>(g.fo);
            const int64_t n = static_cast<int64_t>(g.n);
            T* base = reinterpret_cast<T*>(g.ptr & ~1ull);
            full[j] = valid && (g.ptr & 1ull) && i0 >= 0 && i0 + E <= n;
            if (full[j]) {
                load_vec(base + i0, x[j]);
            } else {
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    const int64_t i = i0 + t;
                    x[j][t] = (valid && i >= 0 && i < n) ? load_one(base + i) : 0.0f;
                }
            }
        }

        if constexpr (UPDATE) {
            float2 acc[V][B][2];
#pragma unroll
            for (int j = 0; j < V; ++j)
#pragma unroll
                for (int b = 0; b < B; ++b) acc[j][b][0] = acc[j][b][1] = make_float2(0.0f, 0.0f);
            const uint32_t K = p.n_seeds;
            if constexpr (Traits<T>::PIPE) {
                // Philox words of seed k + 1 are computed while seed k is transformed
                // and accumulated: the integer-multiply work and the fp32 work of the
                // two halves are independent and interleave in one instruction stream.
                uint4 w[V][B];
                tile_words<V, B>(seed_const(seed_key(p.seeds[0])), blk, w);
                for (uint32_t k = 0; k < K; ++k) {
                    const uint32_t kn = k + 1 < K ? k + 1 : k;
                    uint4 wn[V][B];
                    tile_words<V, B>(seed_const(seed_key(p.seeds[kn])), blk, wn);
                    tile_accumulate<V, B>(w, p.seeds[k].coef, acc);
#pragma unroll
                    for (int j = 0; j < V; ++j)
#pragma unroll
                        for (int b = 0; b < B; ++b) w[j][b] = wn[j][b];
                }
            } else {
                for (uint32_t k = 0; k < K; ++k) {
                    uint4 w[V][B];
                    tile_words<V, B>(seed_const(seed_key(p.seeds[k])), blk, w);
                    tile_accumulate<V, B>(w, p.seeds[k].coef, acc);
                }
            }
#pragma unroll
            for (int j = 0; j < V; ++j)
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    x[j][4 * b + 0] = __fadd_rn(x[j][4 * b + 0], acc[j][b][0].x);
                    x[j][4 * b + 2] = __fadd_rn(x[j][4 * b + 2], acc[j][b][0].y);
                    x[j][4 * b + 1] = __fadd_rn(x[j][4 * b + 1], acc[j][b][1].x);
                    x[j][4 * b + 3] = __fadd_rn(x[j][4 * b + 3], acc[j][b][1].y);
                }
        } else {
            const SeedConst sc = seed_const(seed_key(p.seeds[0]));
            const float2 eps = splat(p.seeds[0].coef);
            uint4 w[V][B];
            tile_words<V, B>(sc, blk, w);
#pragma unroll
            for (int j = 0; j < V; ++j)
#pragma unroll
                for (int b = 0; b < B; ++b) {
                    const GaussPair g = box_muller2(w[j][b]);
                    const float2 ev = fma2<kPackO>(eps, g.even, make_float2(x[j][4 * b + 0], x[j][4 * b + 2]));
                    const float2 od = fma2<kPackO>(eps, g.odd, make_float2(x[j][4 * b + 1], x[j][4 * b + 3]));
                    x[j][4 * b + 0] = ev.x;
                    x[j][4 * b + 2] = ev.y;
                    x[j][4 * b + 1] = od.x;
                    x[j][4 * b + 3] = od.y;
                }
        }

#pragma unroll
        for (int j = 0; j < V; ++j) {
            const uint64_t vi = wt * (32u * V) + 32u * j + lane;
            if (vi >= n_vec) continue;
            const SegParam& g = p.segs[seg[j]];
            T* base = reinterpret_cast<T*>(g.ptr & ~1ull);
            const int64_t i0 = static_cast<int64_t>(blk[j] << 2) - static_cast<int64_t>(g.fo);
            if (full[j]) {
                store_vec(base + i0, x[j]);
            } else {
                const int64_t n = static_cast<int64_t>(g.n);
#pragma unroll
                for (int t = 0; t < E; ++t) {
                    const int64_t i = i0 + t;
                    if (i >= 0 && i < n) store_one(base + i, x[j][t]);
                }
            }
        }
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
constexpr int kKernels = 4;
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
        constexpr uint64_t vec_per_cta = 32ull * Traits<T>::V * (kThreads / 32);
        const uint64_t needed = (p.n_vec + vec_per_cta - 1) / vec_per_cta;
        if (needed < static_cast<uint64_t>(grid)) grid = static_cast<int>(needed);
    }
    kernel<<<grid, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_update(const UpdateParams& p, int dtype, int grid_ctas, cudaStream_t s) {
    if (dtype == kF32) return launch_seeded<float, true>(p, 0, grid_ctas, s);
    return launch_seeded<__nv_bfloat16, true>(p, 1, grid_ctas, s);
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
