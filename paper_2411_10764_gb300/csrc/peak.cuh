// Walk-rate ceiling of the full-table walk (measurement only; peak.cu).
#pragma once

#include "mlt_internal.cuh"

namespace mlt {

// Kernel of depth 1..10 for group 2, 4 or 8 (nullptr otherwise).
using WalkPeakKernelPtr = void (*)(TraverseArgs, int, int, float*);
WalkPeakKernelPtr walk_peak_kernel(int depth, int group);
// Byte offset of its resident trees in shared memory (after the tile of TC
// candidates x F features).
size_t walk_peak_tree_offset(int F, int TC);

}  // namespace mlt
