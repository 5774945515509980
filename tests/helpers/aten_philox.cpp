// Known-answer source for the Philox4x32-10 stream: calls PyTorch's header-only
// at::Philox4_32 engine (it is not copied). Its state maps to the Philox
// counter as (offset lo, offset hi, subsequence lo, subsequence hi) and its key
// is the 64-bit seed, so a block (b, step, sample) under machine id m is
// at::Philox4_32(m, step | sample << 32, b) and its next four outputs.
#include <ATen/core/PhiloxRNGEngine.h>
#include <cstdint>

extern "C" void aten_philox_blocks(uint64_t seed, uint64_t subsequence, uint64_t first_offset,
                                   uint64_t n_blocks, uint32_t* out) {
    for (uint64_t i = 0; i < n_blocks; ++i) {
        at::Philox4_32 engine(seed, subsequence, first_offset + i);
        for (int w = 0; w < 4; ++w) out[4 * i + w] = engine();
    }
}

// The first `rounds` Philox rounds of counter (offset lo, offset hi, subsequence lo,
// subsequence hi) under key `seed`: at::Philox4_32 takes the round count per draw.
extern "C" void aten_philox_rounds(uint64_t seed, uint64_t subsequence, uint64_t offset,
                                   int rounds, uint32_t* out) {
    at::Philox4_32 engine(seed, subsequence, offset);
    for (int w = 0; w < 4; ++w) out[w] = engine(rounds);
}
