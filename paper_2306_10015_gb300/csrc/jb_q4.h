// jb_q4.h -- the unit shape of the 4-bit perturbation kernel, shared by the kernel
// (jb_q4.cu) and the host code that numbers the units of each tensor (jb_capi.cpp).
#pragma once

namespace jb {

constexpr int kQ4Epl = 32;                     // elements per lane and unit
constexpr int kQ4UnitsPerBlock = 64 / kQ4Epl;  // units per 64-element scale block

}  // namespace jb
