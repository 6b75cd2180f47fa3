// Internal declarations of the temporal module (Section 3.2, Eq. 12-13); not part of the public ABI.
#pragma once

#include "hg_internal.cuh"

namespace hg {

// Largest context window the kernels accept.
constexpr int kTemporalMaxW = 8;

}  // namespace hg
