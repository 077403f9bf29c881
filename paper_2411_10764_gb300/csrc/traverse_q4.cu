// Full-table walk kernels with 4 tree groups per CTA (stored and decoded
// features): instantiated apart so the build compiles them in parallel.
#include "walk.cuh"

namespace mlt {

FullKernelPtr full_kernel_q4(int depth, int group) { return walk::full_kernel_q<4>(depth, group); }
FullDecKernelPtr full_dec_kernel_q4(int depth, int group) { return walk::full_dec_kernel_q<4>(depth, group); }

}  // namespace mlt
