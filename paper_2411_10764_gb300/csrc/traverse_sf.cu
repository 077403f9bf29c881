// Full-table walk kernels with one tree group and the barrier-free chunk
// pipeline (stored and decoded features): instantiated apart so the build
// compiles them in parallel.
#include "walk.cuh"

namespace mlt {

FullKernelPtr full_kernel_sf(int depth, int group) { return walk::full_kernel_q<0>(depth, group); }
FullDecKernelPtr full_dec_kernel_sf(int depth, int group) { return walk::full_dec_kernel_q<0>(depth, group); }

}  // namespace mlt
