// jb_internal.h -- launch descriptors shared by the C ABI (jb_capi.cpp) and
// the kernels (jb_kernels.cu). Not part of the public interface.
//
// A launch carries its whole work description in the kernel parameter space
// (up to 32,764 bytes on sm_70 and later): the K (seed, coefficient) pairs are
// read with warp-uniform indices from the constant bank, and the segment table
// maps a flat "vector" index to a tensor. A vector is 16 bytes of one segment
// whose elements are aligned to Philox blocks in global index: 4 fp32 or 8
// bf16 elements. Segment s owns the global vectors floor(fo / E) ..
// ceil((fo + n) / E) - 1; its first one is launch vector vec0.
#pragma once
#include <cstdint>

#include <cuda_runtime.h>

namespace jb {

#ifndef JB_THREADS
#define JB_THREADS 512
#endif
constexpr int kThreads = JB_THREADS;   // threads per CTA
constexpr int kMaxSeedsPerLaunch = 512;
constexpr int kMaxSegsUpdate = 700;    // 16 + 512 * 20 + 700 * 32 bytes
constexpr int kMaxSegsPerturb = 1000;  // 16 + 24 + 1000 * 32 bytes

struct SeedParam {
    uint32_t k0, k1;        // machine id (lo, hi)
    uint32_t step, sample;  // counter words 2 and 3
    float coef;             // c_k (update) or eps (perturb)
};

struct SegParam {
    uint64_t ptr;   // device address; bit 0 set when the 16-byte vector path applies
    uint64_t fo;    // global index of element 0
    uint64_t n;     // elements
    uint64_t vec0;  // first launch vector of this segment
};

template <int MAXK, int MAXS>
struct LaunchParams {
    uint32_t n_seeds;
    uint32_t n_segs;
    uint64_t n_vec;  // vectors in this launch
    SeedParam seeds[MAXK];
    SegParam segs[MAXS];
};

using UpdateParams = LaunchParams<kMaxSeedsPerLaunch, kMaxSegsUpdate>;
using PerturbParams = LaunchParams<1, kMaxSegsPerturb>;

static_assert(sizeof(UpdateParams) <= 32764, "update launch exceeds the parameter space");
static_assert(sizeof(PerturbParams) <= 32764, "perturb launch exceeds the parameter space");

// Generalised update: reads segment `ptr`, writes segment `dst` (and `ptr` too when
// write_src), and applies the seeds in groups, rounding to the storage type after
// each group: group g covers seeds [group_end[g - 1], group_end[g]).
constexpr int kMaxGroupsPerLaunch = 512;
constexpr int kMaxSegsGeneral = 512;

struct SegParamOut {
    uint64_t ptr;   // source; bit 0 set when source and destination take the vector path
    uint64_t dst;   // destination
    uint64_t fo;
    uint64_t n;
    uint64_t vec0;
};

struct GeneralParams {
    uint32_t n_seeds;
    uint32_t n_segs;
    uint64_t n_vec;
    uint32_t n_groups;
    uint32_t write_src;
    SeedParam seeds[kMaxSeedsPerLaunch];
    uint16_t group_end[kMaxGroupsPerLaunch];
    SegParamOut segs[kMaxSegsGeneral];
};

static_assert(sizeof(GeneralParams) <= 32764, "general launch exceeds the parameter space");

// 4-bit weights: codes (two per byte, element 2i in the low nibble) and one fp32
// scale per 64 elements. Work unit: 16 elements (8 code bytes); a segment owns
// units [unit0, unit0 + ceil(n / 64) * 4), so a 64-element block is always four
// consecutive units, handled by four consecutive lanes.
constexpr int kMaxSegsQ4 = 800;

struct SegParamQ4 {
    uint64_t codes;  // device address, 8-byte aligned
    uint64_t scale;  // device address of the fp32 scales
    uint64_t fo;     // global index of element 0 (a multiple of 4)
    uint64_t n;
    uint64_t unit0;
};

struct Q4Params {
    SeedParam seed;  // coef = eps
    uint32_t n_segs;
    uint64_t n_units;
    SegParamQ4 segs[kMaxSegsQ4];
};

static_assert(sizeof(Q4Params) <= 32764, "4-bit launch exceeds the parameter space");

cudaError_t launch_q4_perturb(const Q4Params& p, int grid_ctas, cudaStream_t s);
void q4_levels_host(float out[16]);

enum DType { kF32 = 0, kBF16 = 1 };

// Launchers (jb_kernels.cu). grid_ctas <= 0 selects the persistent grid.
cudaError_t launch_update(const UpdateParams& p, int dtype, int grid_ctas, cudaStream_t s);
cudaError_t launch_perturb(const PerturbParams& p, int dtype, int grid_ctas, cudaStream_t s);
cudaError_t launch_general(const GeneralParams& p, int dtype, int grid_ctas, cudaStream_t s);
cudaError_t launch_checksum(const PerturbParams& p, int dtype, unsigned long long* out,
                            int grid_ctas, cudaStream_t s);
cudaError_t launch_debug_philox(SeedParam seed, uint64_t first_block, uint64_t n_blocks,
                                uint32_t* out, cudaStream_t s);
cudaError_t launch_debug_philox_fold(SeedParam seed, uint64_t first_block, uint64_t n_blocks,
                                     uint32_t* out, cudaStream_t s);
cudaError_t launch_debug_gaussian(SeedParam seed, uint64_t first, uint64_t n, float* out,
                                  cudaStream_t s);
cudaError_t launch_debug_box_muller(const uint32_t* words, uint64_t n_pairs, float* out,
                                    cudaStream_t s);

}  // namespace jb
