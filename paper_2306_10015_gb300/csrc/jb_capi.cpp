// jb_capi.cpp -- the C ABI of libjb (declared in include/jb.h).
//
// Host side of the hot path: argument checks, the canonical (machine id,
// step, sample id) order of the pairs (Section 2: gradients are applied in
// machine-timestamp order), the per-pair coefficients c_k = -lr deq(q_k) /
// denom (Algorithm 1: minus gradient times learning rate over the number of
// gradients), the one-byte code (Section 3, Training Speed), and the packing of
// segments and pairs into kernel launches. Every element-wise step runs in the CUDA kernels.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <vector>

#include "jb.h"
#include "jb_internal.h"
#include "jb_q4.h"

#define JB_EXPORT extern "C" __attribute__((visibility("default")))

namespace {

constexpr uint64_t kMaxIndex = 1ull << 62;  // global element indices stay below this

struct Seg {
    uint64_t ptr, fo, n;
};

size_t elem_size(int dtype) { return dtype == JB_F32 ? 4 : 2; }

// [p, p + n * es) fits in the address space (written so that n * es cannot wrap).
bool range_fits(uint64_t p, uint64_t n, uint64_t es) { return n <= (UINT64_MAX - p) / es; }

// Runs an entry point's body; a host allocation failure (or any other C++
// exception) becomes a status instead of crossing the C interface.
template <typename F>
int guarded(F&& body) noexcept {
    try {
        return body();
    } catch (const std::bad_alloc&) {
        return JB_ERR_NO_MEMORY;
    } catch (...) {
        return JB_ERR_INVALID_ARG;
    }
}
int elems_per_vec(int dtype) { return dtype == JB_F32 ? 4 : 8; }

// Checks the segment table; drops empty segments. Overlap in memory or in
// global index is an argument error.
int collect_segments(const jb_segment* segs, int n_segs, int dtype, std::vector<Seg>& out) {
    if (dtype != JB_F32 && dtype != JB_BF16) return JB_ERR_UNSUPPORTED_DTYPE;
    if (n_segs < 0 || (n_segs > 0 && segs == nullptr)) return JB_ERR_INVALID_ARG;
    const uint64_t es = elem_size(dtype);
    out.clear();
    out.reserve(static_cast<size_t>(n_segs));
    for (int i = 0; i < n_segs; ++i) {
        const jb_segment& s = segs[i];
        if (s.numel == 0) continue;
        const uint64_t p = reinterpret_cast<uint64_t>(s.ptr);
        if (p == 0) return JB_ERR_INVALID_ARG;
        if (p % es != 0) return JB_ERR_MISALIGNED;
        if (s.numel > kMaxIndex || s.flat_offset > kMaxIndex - s.numel) return JB_ERR_INVALID_ARG;
        if (!range_fits(p, s.numel, es)) return JB_ERR_INVALID_ARG;
        out.push_back({p, s.flat_offset, s.numel});
    }
    std::vector<Seg> by_fo(out), by_ptr(out);
    std::sort(by_fo.begin(), by_fo.end(), [](const Seg& a, const Seg& b) { return a.fo < b.fo; });
    for (size_t i = 1; i < by_fo.size(); ++i)
        if (by_fo[i - 1].fo + by_fo[i - 1].n > by_fo[i].fo) return JB_ERR_INVALID_ARG;
    std::sort(by_ptr.begin(), by_ptr.end(), [](const Seg& a, const Seg& b) { return a.ptr < b.ptr; });
    for (size_t i = 1; i < by_ptr.size(); ++i)
        if (by_ptr[i - 1].ptr + by_ptr[i - 1].n * es > by_ptr[i].ptr) return JB_ERR_INVALID_ARG;
    return JB_OK;
}

// Fills params.segs / n_segs / n_vec with segments [first, first + count).
template <typename P>
void pack_segments(const std::vector<Seg>& segs, size_t first, size_t count, int dtype, P& params) {
    const uint64_t E = static_cast<uint64_t>(elems_per_vec(dtype));
    const uint64_t es = elem_size(dtype);
    uint64_t vec = 0;
    for (size_t i = 0; i < count; ++i) {
        const Seg& s = segs[first + i];
        jb::SegParam& g = params.segs[i];
        const uint64_t v_begin = s.fo / E;
        const uint64_t v_end = (s.fo + s.n + E - 1) / E;
        // 16-byte vectors of the segment line up with element groups whose global
        // index is a multiple of E iff ptr - fo * sizeof(T) is 16-byte aligned.
        const bool aligned = ((s.ptr - s.fo * es) & 15ull) == 0;
        g.ptr = s.ptr | (aligned ? 1ull : 0ull);
        g.fo = s.fo;
        g.n = s.n;
        g.vec0 = vec;
        vec += v_end - v_begin;
    }
    params.n_segs = static_cast<uint32_t>(count);
    params.n_vec = vec;
}

jb::SeedParam seed_param(const jb_seed& s, float coef) {
    jb::SeedParam p;
    p.k0 = static_cast<uint32_t>(s.machine_id);
    p.k1 = static_cast<uint32_t>(s.machine_id >> 32);
    p.step = s.step;
    p.sample = s.sample_id;
    p.coef = coef;
    return p;
}

bool seed_less(const jb_seed& a, const jb_seed& b) {
    if (a.machine_id != b.machine_id) return a.machine_id < b.machine_id;
    if (a.step != b.step) return a.step < b.step;
    return a.sample_id < b.sample_id;
}

bool seed_equal(const jb_seed& a, const jb_seed& b) {
    return a.machine_id == b.machine_id && a.step == b.step && a.sample_id == b.sample_id;
}

double dequantize(int8_t q, double qscale) {
    int m = q < 0 ? -static_cast<int>(q) : static_cast<int>(q);
    if (m > 127) m = 127;
    const double v = std::expm1(static_cast<double>(m) / qscale);
    return q < 0 ? -v : v;
}

// libjb links the CUDA runtime statically: its last-error state is its own, so the
// errors of a caller's runtime (torch's, say) are neither seen nor cleared here. A
// failed call of this library's is cleared from that state (cudaGetLastError) so that
// it cannot be reported again by a later, unrelated call.
int cuda_status(cudaError_t e) {
    if (e == cudaSuccess) return JB_OK;
    (void)cudaGetLastError();
    return JB_ERR_CUDA;
}

int perturb_impl(const jb_segment* segs, int n_segs, int dtype, jb_seed seed, float eps,
                 int grid_ctas, cudaStream_t stream) {
    std::vector<Seg> v;
    int rc = collect_segments(segs, n_segs, dtype, v);
    if (rc != JB_OK) return rc;
    if (!std::isfinite(eps)) return JB_ERR_INVALID_ARG;
    if (v.empty()) return JB_OK;
    static thread_local jb::PerturbParams params;  // ~32 KB: keep it off the stack
    params.n_seeds = 1;
    params.seeds[0] = seed_param(seed, eps);
    for (size_t first = 0; first < v.size(); first += jb::kMaxSegsPerturb) {
        const size_t count = std::min<size_t>(jb::kMaxSegsPerturb, v.size() - first);
        pack_segments(v, first, count, dtype, params);
        rc = cuda_status(jb::launch_perturb(params, dtype, grid_ctas, stream));
        if (rc != JB_OK) return rc;
    }
    return JB_OK;
}

int update_impl(const jb_segment* segs, int n_segs, int dtype, const jb_seed* seeds,
                const int8_t* q, int K, float lr, float denom, float qscale, int grid_ctas,
                cudaStream_t stream) {
    std::vector<Seg> v;
    int rc = collect_segments(segs, n_segs, dtype, v);
    if (rc != JB_OK) return rc;
    if (K < 0 || (K > 0 && (seeds == nullptr || q == nullptr))) return JB_ERR_INVALID_ARG;
    if (!std::isfinite(lr) || !std::isfinite(denom) || denom == 0.0f || !std::isfinite(qscale) ||
        !(qscale > 0.0f))
        return JB_ERR_INVALID_ARG;
    if (K > jb::kMaxSeedsPerLaunch) return JB_ERR_TOO_MANY_SEEDS;
    if (K == 0) return JB_OK;

    // Canonical order: ascending (machine id, step, sample id).
    std::vector<int> order(static_cast<size_t>(K));
    for (int k = 0; k < K; ++k) order[k] = k;
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return seed_less(seeds[a], seeds[b]); });
    for (int k = 1; k < K; ++k)
        if (seed_equal(seeds[order[k - 1]], seeds[order[k]])) return JB_ERR_DUPLICATE_SEED;

    static thread_local jb::UpdateParams params;
    params.n_seeds = static_cast<uint32_t>(K);
    for (int k = 0; k < K; ++k) {
        const int i = order[k];
        const double c = -static_cast<double>(lr) * dequantize(q[i], static_cast<double>(qscale)) /
                         static_cast<double>(denom);
        const float cf = static_cast<float>(c);
        if (!std::isfinite(cf)) return JB_ERR_RANGE;
        params.seeds[k] = seed_param(seeds[i], cf);
    }
    if (v.empty()) return JB_OK;
    for (size_t first = 0; first < v.size(); first += jb::kMaxSegsUpdate) {
        const size_t count = std::min<size_t>(jb::kMaxSegsUpdate, v.size() - first);
        pack_segments(v, first, count, dtype, params);
        rc = cuda_status(jb::launch_update(params, dtype, grid_ctas, stream));
        if (rc != JB_OK) return rc;
    }
    return JB_OK;
}

// Destination table for src: same numel and flat offsets, element-aligned; each
// destination either is its source or overlaps no source and no other destination.
int collect_destinations(const jb_segment* src, const jb_segment* dst, int n_segs, int dtype,
                         std::vector<uint64_t>& dptr) {
    if (n_segs > 0 && dst == nullptr) return JB_ERR_INVALID_ARG;
    const uint64_t es = elem_size(dtype);
    struct Iv { uint64_t a, b; int owner; bool is_dst; };
    std::vector<Iv> iv;
    dptr.clear();
    for (int i = 0; i < n_segs; ++i) {
        if (src[i].numel == 0) {
            if (dst[i].numel != 0) return JB_ERR_INVALID_ARG;
            continue;
        }
        if (dst[i].numel != src[i].numel || dst[i].flat_offset != src[i].flat_offset)
            return JB_ERR_INVALID_ARG;
        const uint64_t p = reinterpret_cast<uint64_t>(dst[i].ptr);
        if (p == 0) return JB_ERR_INVALID_ARG;
        if (p % es != 0) return JB_ERR_MISALIGNED;
        if (!range_fits(p, dst[i].numel, es)) return JB_ERR_INVALID_ARG;
        dptr.push_back(p);
        const uint64_t sp = reinterpret_cast<uint64_t>(src[i].ptr);
        iv.push_back({sp, sp + src[i].numel * es, i, false});
        if (p != sp) iv.push_back({p, p + src[i].numel * es, i, true});
    }
    std::sort(iv.begin(), iv.end(), [](const Iv& x, const Iv& y) { return x.a < y.a; });
    for (size_t i = 1; i < iv.size(); ++i)
        if (iv[i - 1].b > iv[i].a) return JB_ERR_INVALID_ARG;
    return JB_OK;
}

// Shared by jb_apply_updates_from and jb_replay_updates: groups of pairs applied in
// order, each group in canonical order with its own lr and denom, one rounding to
// the storage type per group.
int general_impl(const jb_segment* segs, const jb_segment* dsts, int n_segs, int dtype,
                 const jb_seed* seeds, const int8_t* q, const int* group_sizes, int n_groups,
                 const float* lr, const float* denom, float qscale, int write_src, int grid_ctas,
                 cudaStream_t stream) {
    std::vector<Seg> v;
    int rc = collect_segments(segs, n_segs, dtype, v);
    if (rc != JB_OK) return rc;
    std::vector<uint64_t> dptr;
    const bool out_of_place = dsts != nullptr;
    if (out_of_place) {
        rc = collect_destinations(segs, dsts, n_segs, dtype, dptr);
        if (rc != JB_OK) return rc;
    } else {
        for (const Seg& g : v) dptr.push_back(g.ptr);
    }
    if (n_groups < 0 || (n_groups > 0 && (group_sizes == nullptr || lr == nullptr || denom == nullptr)))
        return JB_ERR_INVALID_ARG;
    if (!std::isfinite(qscale) || !(qscale > 0.0f)) return JB_ERR_INVALID_ARG;
    long long total = 0;
    for (int g = 0; g < n_groups; ++g) {
        if (group_sizes[g] < 0) return JB_ERR_INVALID_ARG;
        if (group_sizes[g] > jb::kMaxSeedsPerLaunch) return JB_ERR_TOO_MANY_SEEDS;
        if (!std::isfinite(lr[g]) || !std::isfinite(denom[g]) || denom[g] == 0.0f)
            return JB_ERR_INVALID_ARG;
        total += group_sizes[g];
    }
    if (total > 0 && (seeds == nullptr || q == nullptr)) return JB_ERR_INVALID_ARG;

    // every group in canonical order, with its coefficients
    std::vector<jb::SeedParam> all(static_cast<size_t>(total));
    std::vector<int> sizes;
    long long base = 0;
    for (int g = 0; g < n_groups; ++g) {
        const int K = group_sizes[g];
        std::vector<int> order(static_cast<size_t>(K));
        for (int k = 0; k < K; ++k) order[k] = static_cast<int>(base) + k;
        std::stable_sort(order.begin(), order.end(),
                         [&](int a, int b) { return seed_less(seeds[a], seeds[b]); });
        for (int k = 1; k < K; ++k)
            if (seed_equal(seeds[order[k - 1]], seeds[order[k]])) return JB_ERR_DUPLICATE_SEED;
        for (int k = 0; k < K; ++k) {
            const int i = order[k];
            const double c = -static_cast<double>(lr[g]) * dequantize(q[i], static_cast<double>(qscale)) /
                             static_cast<double>(denom[g]);
            const float cf = static_cast<float>(c);
            if (!std::isfinite(cf)) return JB_ERR_RANGE;
            all[static_cast<size_t>(base + k)] = seed_param(seeds[i], cf);
        }
        base += K;
        if (K > 0) sizes.push_back(K);  // an empty group changes nothing
    }
    if (v.empty()) return JB_OK;
    if (sizes.empty()) {
        if (!out_of_place) return JB_OK;
        sizes.clear();  // a pure copy: one launch with no group
    }

    static thread_local jb::GeneralParams params;
    const uint64_t E = static_cast<uint64_t>(elems_per_vec(dtype));
    const uint64_t es = elem_size(dtype);
    // groups in launches of at most kMaxSeedsPerLaunch pairs / kMaxGroupsPerLaunch groups;
    // after the first launch the destination holds the running value
    size_t g0 = 0;
    long long s0 = 0;
    bool first = true;
    do {
        size_t g1 = g0;
        long long n = 0;
        while (g1 < sizes.size() && g1 - g0 < static_cast<size_t>(jb::kMaxGroupsPerLaunch) &&
               n + sizes[g1] <= jb::kMaxSeedsPerLaunch)
            n += sizes[g1++];
        params.n_seeds = static_cast<uint32_t>(n);
        params.n_groups = static_cast<uint32_t>(g1 - g0);
        long long acc = 0;
        for (size_t g = g0; g < g1; ++g) {
            acc += sizes[g];
            params.group_end[g - g0] = static_cast<uint16_t>(acc);
        }
        for (long long k = 0; k < n; ++k) params.seeds[k] = all[static_cast<size_t>(s0 + k)];
        const bool last = g1 >= sizes.size();
        // write_src comes with one group only (jb_apply_updates_from): one launch round
        params.write_src = (write_src && last) ? 1u : 0u;
        for (size_t first_seg = 0; first_seg < v.size(); first_seg += jb::kMaxSegsGeneral) {
            const size_t count = std::min<size_t>(jb::kMaxSegsGeneral, v.size() - first_seg);
            uint64_t vec = 0;
            for (size_t i = 0; i < count; ++i) {
                const Seg& sg = v[first_seg + i];
                const uint64_t src_ptr = first ? sg.ptr : dptr[first_seg + i];
                const uint64_t dst_ptr = dptr[first_seg + i];
                jb::SegParamOut& g = params.segs[i];
                const bool aligned = ((src_ptr - sg.fo * es) & 15ull) == 0 &&
                                     ((dst_ptr - sg.fo * es) & 15ull) == 0;
                g.ptr = src_ptr | (aligned ? 1ull : 0ull);
                g.dst = dst_ptr;
                g.fo = sg.fo;
                g.n = sg.n;
                g.vec0 = vec;
                vec += (sg.fo + sg.n + E - 1) / E - sg.fo / E;
            }
            params.n_segs = static_cast<uint32_t>(count);
            params.n_vec = vec;
            rc = cuda_status(jb::launch_general(params, dtype, grid_ctas, stream));
            if (rc != JB_OK) return rc;
        }
        s0 += n;
        g0 = g1;
        first = false;
    } while (g0 < sizes.size());
    return JB_OK;
}

}  // namespace

JB_EXPORT int jb_apply_updates_from(const jb_segment* src, const jb_segment* dst, int n_segs,
                                    int dtype, const jb_seed* seeds, const int8_t* q, int K,
                                    float lr, float denom, float qscale, int write_src,
                                    struct CUstream_st* stream) {
    if (dst == nullptr && n_segs > 0) return JB_ERR_INVALID_ARG;
    if (K < 0) return JB_ERR_INVALID_ARG;
    return guarded([&] {
        return general_impl(src, dst, n_segs, dtype, seeds, q, &K, 1, &lr, &denom, qscale, write_src,
                            0, stream);
    });
}

JB_EXPORT int jb_replay_updates(const jb_segment* segs, int n_segs, int dtype, const jb_seed* seeds,
                                const int8_t* q, const int* step_sizes, int n_steps,
                                const float* lr, const float* denom, float qscale,
                                struct CUstream_st* stream) {
    return guarded([&] {
        return general_impl(segs, nullptr, n_segs, dtype, seeds, q, step_sizes, n_steps, lr, denom,
                            qscale, 0, 0, stream);
    });
}

JB_EXPORT int jb_perturb(const jb_segment* segs, int n_segs, int dtype, jb_seed seed, float eps,
                         struct CUstream_st* stream) {
    return guarded([&] { return perturb_impl(segs, n_segs, dtype, seed, eps, 0, stream); });
}

JB_EXPORT int jb_perturb_with_grid(const jb_segment* segs, int n_segs, int dtype, jb_seed seed,
                                   float eps, int grid_ctas, struct CUstream_st* stream) {
    return guarded([&] { return perturb_impl(segs, n_segs, dtype, seed, eps, grid_ctas, stream); });
}

JB_EXPORT int jb_apply_updates(const jb_segment* segs, int n_segs, int dtype, const jb_seed* seeds,
                               const int8_t* q, int K, float lr, float denom, float qscale,
                               struct CUstream_st* stream) {
    return guarded([&] { return update_impl(segs, n_segs, dtype, seeds, q, K, lr, denom, qscale, 0, stream); });
}

JB_EXPORT int jb_apply_updates_with_grid(const jb_segment* segs, int n_segs, int dtype,
                                         const jb_seed* seeds, const int8_t* q, int K, float lr,
                                         float denom, float qscale, int grid_ctas,
                                         struct CUstream_st* stream) {
    return guarded(
        [&] { return update_impl(segs, n_segs, dtype, seeds, q, K, lr, denom, qscale, grid_ctas, stream); });
}

namespace {
int checksum_impl(const jb_segment* segs, int n_segs, int dtype, uint64_t* d_out, int grid_ctas,
                  cudaStream_t stream) {
    std::vector<Seg> v;
    int rc = collect_segments(segs, n_segs, dtype, v);
    if (rc != JB_OK) return rc;
    if (d_out == nullptr) return JB_ERR_INVALID_ARG;
    if (reinterpret_cast<uint64_t>(d_out) & 7ull) return JB_ERR_MISALIGNED;
    rc = cuda_status(cudaMemsetAsync(d_out, 0, sizeof(uint64_t), stream));
    if (rc != JB_OK) return rc;
    static thread_local jb::PerturbParams params;
    params.n_seeds = 0;
    for (size_t first = 0; first < v.size(); first += jb::kMaxSegsPerturb) {
        const size_t count = std::min<size_t>(jb::kMaxSegsPerturb, v.size() - first);
        pack_segments(v, first, count, dtype, params);
        rc = cuda_status(jb::launch_checksum(params, dtype, reinterpret_cast<unsigned long long*>(d_out),
                                             grid_ctas, stream));
        if (rc != JB_OK) return rc;
    }
    return JB_OK;
}
}  // namespace

JB_EXPORT int jb_checksum(const jb_segment* segs, int n_segs, int dtype, uint64_t* d_out,
                          struct CUstream_st* stream) {
    return guarded([&] { return checksum_impl(segs, n_segs, dtype, d_out, 0, stream); });
}

JB_EXPORT int jb_checksum_with_grid(const jb_segment* segs, int n_segs, int dtype, uint64_t* d_out,
                                    int grid_ctas, struct CUstream_st* stream) {
    return guarded([&] { return checksum_impl(segs, n_segs, dtype, d_out, grid_ctas, stream); });
}

namespace {
int perturb_q4_impl(const jb_q4_segment* segs, int n_segs, jb_seed seed, float eps, cudaStream_t stream) {
    if (n_segs < 0 || (n_segs > 0 && segs == nullptr)) return JB_ERR_INVALID_ARG;
    if (!std::isfinite(eps)) return JB_ERR_INVALID_ARG;
    struct Q { uint64_t codes, scale, fo, n; };
    std::vector<Q> v;
    struct Iv { uint64_t a, b; };
    std::vector<Iv> mem, idx;
    for (int i = 0; i < n_segs; ++i) {
        const jb_q4_segment& g = segs[i];
        if (g.numel == 0) continue;
        const uint64_t c = reinterpret_cast<uint64_t>(g.codes), sp = reinterpret_cast<uint64_t>(g.scale);
        if (c == 0 || sp == 0) return JB_ERR_INVALID_ARG;
        if ((c & 7ull) || (sp & 3ull) || (g.flat_offset & 3ull)) return JB_ERR_MISALIGNED;
        if (g.numel > kMaxIndex || g.flat_offset > kMaxIndex - g.numel) return JB_ERR_INVALID_ARG;
        const uint64_t nb = (g.numel + 1) / 2, ns = 4 * ((g.numel + 63) / 64);
        if (c > UINT64_MAX - nb || sp > UINT64_MAX - ns) return JB_ERR_INVALID_ARG;
        v.push_back({c, sp, g.flat_offset, g.numel});
        mem.push_back({c, c + nb});
        mem.push_back({sp, sp + ns});
        idx.push_back({g.flat_offset, g.flat_offset + g.numel});
    }
    for (auto* list : {&mem, &idx}) {
        std::sort(list->begin(), list->end(), [](const Iv& x, const Iv& y) { return x.a < y.a; });
        for (size_t i = 1; i < list->size(); ++i)
            if ((*list)[i - 1].b > (*list)[i].a) return JB_ERR_INVALID_ARG;
    }
    if (v.empty()) return JB_OK;
    static thread_local jb::Q4Params params;
    params.seed = seed_param(seed, eps);
    for (size_t first = 0; first < v.size(); first += jb::kMaxSegsQ4) {
        const size_t count = std::min<size_t>(jb::kMaxSegsQ4, v.size() - first);
        uint64_t unit = 0;
        for (size_t i = 0; i < count; ++i) {
            const Q& q = v[first + i];
            jb::SegParamQ4& g = params.segs[i];
            g.codes = q.codes;
            g.scale = q.scale;
            g.fo = q.fo;
            g.n = q.n;
            g.unit0 = unit;
            unit += jb::kQ4UnitsPerBlock * ((q.n + 63) / 64);  // whole 64-element blocks
        }
        params.n_segs = static_cast<uint32_t>(count);
        params.n_units = unit;
        const int rc = cuda_status(jb::launch_q4_perturb(params, 0, stream));
        if (rc != JB_OK) return rc;
    }
    return JB_OK;
}
}  // namespace

JB_EXPORT int jb_perturb_q4(const jb_q4_segment* segs, int n_segs, jb_seed seed, float eps,
                            struct CUstream_st* stream) {
    return guarded([&] { return perturb_q4_impl(segs, n_segs, seed, eps, stream); });
}

JB_EXPORT int jb_q4_levels(float* out) {
    if (out == nullptr) return JB_ERR_INVALID_ARG;
    jb::q4_levels_host(out);
    return JB_OK;
}

JB_EXPORT int jb_quantize_grad(double g, float qscale, int8_t* out) {
    if (out == nullptr || !std::isfinite(qscale) || !(qscale > 0.0f)) return JB_ERR_INVALID_ARG;
    if (std::isnan(g)) {
        *out = 0;
        return JB_OK;
    }
    double mag = std::isinf(g) ? 127.0
                               : std::round(static_cast<double>(qscale) * std::log1p(std::fabs(g)));
    if (mag > 127.0) mag = 127.0;
    const int m = static_cast<int>(mag);
    *out = static_cast<int8_t>(g < 0 ? -m : m);
    return JB_OK;
}

JB_EXPORT int jb_dequantize_grad(int8_t q, float qscale, float* out) {
    if (out == nullptr || !std::isfinite(qscale) || !(qscale > 0.0f)) return JB_ERR_INVALID_ARG;
    *out = static_cast<float>(dequantize(q, static_cast<double>(qscale)));
    return JB_OK;
}

JB_EXPORT int jb_max_seeds_per_call(void) { return jb::kMaxSeedsPerLaunch; }

JB_EXPORT const char* jb_status_string(int status) {
    switch (status) {
        case JB_OK: return "ok";
        case JB_ERR_INVALID_ARG: return "invalid argument";
        case JB_ERR_UNSUPPORTED_DTYPE: return "unsupported dtype (use JB_F32 or JB_BF16)";
        case JB_ERR_MISALIGNED: return "segment pointer not aligned to its element size";
        case JB_ERR_DUPLICATE_SEED: return "duplicate (machine_id, step, sample_id) seed";
        case JB_ERR_CUDA: return "CUDA runtime or launch error";
        case JB_ERR_RANGE: return "update coefficient not finite in fp32";
        case JB_ERR_TOO_MANY_SEEDS: return "more seeds than one call accepts";
        case JB_ERR_NO_MEMORY: return "host memory allocation failed";
        default: return "unknown status";
    }
}

JB_EXPORT int jb_debug_philox(jb_seed seed, uint64_t first_block, uint64_t n_blocks, uint32_t* d_out,
                              struct CUstream_st* stream) {
    if (n_blocks > 0 && d_out == nullptr) return JB_ERR_INVALID_ARG;
    if (n_blocks > (1ull << 38)) return JB_ERR_INVALID_ARG;
    if (reinterpret_cast<uint64_t>(d_out) & 15ull) return JB_ERR_MISALIGNED;  // one 16-byte store per block
    return cuda_status(jb::launch_debug_philox(seed_param(seed, 0.0f), first_block, n_blocks, d_out,
                                               stream));
}

JB_EXPORT int jb_debug_philox_fold(jb_seed seed, uint64_t first_block, uint64_t n_blocks,
                                   uint32_t* d_out, struct CUstream_st* stream) {
    if (d_out == nullptr) return JB_ERR_INVALID_ARG;
    if (n_blocks > (1ull << 46) || first_block > (1ull << 60)) return JB_ERR_INVALID_ARG;
    if (reinterpret_cast<uint64_t>(d_out) & 3ull) return JB_ERR_MISALIGNED;
    return cuda_status(jb::launch_debug_philox_fold(seed_param(seed, 0.0f), first_block, n_blocks,
                                                    d_out, stream));
}

JB_EXPORT int jb_debug_gaussian(jb_seed seed, uint64_t first_elem, uint64_t n, float* d_out,
                                struct CUstream_st* stream) {
    if (n > 0 && d_out == nullptr) return JB_ERR_INVALID_ARG;
    if (n > (1ull << 38) || first_elem > kMaxIndex - n) return JB_ERR_INVALID_ARG;
    if (reinterpret_cast<uint64_t>(d_out) & 3ull) return JB_ERR_MISALIGNED;
    return cuda_status(jb::launch_debug_gaussian(seed_param(seed, 0.0f), first_elem, n, d_out, stream));
}

JB_EXPORT int jb_debug_box_muller(const uint32_t* d_words, uint64_t n_pairs, float* d_out,
                                  struct CUstream_st* stream) {
    if (n_pairs > 0 && (d_words == nullptr || d_out == nullptr)) return JB_ERR_INVALID_ARG;
    if (n_pairs > (1ull << 38)) return JB_ERR_INVALID_ARG;
    if ((reinterpret_cast<uint64_t>(d_words) | reinterpret_cast<uint64_t>(d_out)) & 3ull)
        return JB_ERR_MISALIGNED;
    return cuda_status(jb::launch_debug_box_muller(d_words, n_pairs, d_out, stream));
}
