// Tree-walk kernels over half tables (binary16 thresholds, leaves and staged
// features; the tolerance-checked variant of the screening walk): depth
// 1..10, 2, 4 or 8 trees in flight.
#include "walk.cuh"

namespace mlt {

FullKernelPtr half_kernel(int depth, int group, bool sync_free) {
  if (sync_free)
    return group == 8   ? walk::half_kernel_for<8, 0>(depth)
           : group == 4 ? walk::half_kernel_for<4, 0>(depth)
           : group == 2 ? walk::half_kernel_for<2, 0>(depth)
                        : nullptr;
  return group == 8   ? walk::half_kernel_for<8, 1>(depth)
         : group == 4 ? walk::half_kernel_for<4, 1>(depth)
         : group == 2 ? walk::half_kernel_for<2, 1>(depth)
                      : nullptr;
}

}  // namespace mlt
