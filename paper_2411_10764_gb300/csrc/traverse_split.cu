// Tree-walk kernels over split tables (models deeper than a full table
// holds: each tree's first H levels stream through shared memory, the rest
// is read from L2), stored features.  XGBoost gbtree prediction (Sec. 3,
// Table 3) for the unbalanced deep ensembles of the skewed workload.
#include "walk.cuh"

namespace mlt {
namespace {

template <int SH, int G, int QS>
__global__ void __launch_bounds__(QS == 8 ? 1024 : 512, 1) k_traverse_split(const __grid_constant__ TraverseArgs a) {
  walk::traverse_full_body<1, G, QS, false, SH>(a, nullptr);
}

template <int SH, int G>
FullKernelPtr split_for_q(int q) {
  switch (q) {
    case 0: return k_traverse_split<SH, G, 0>;
    case 1: return k_traverse_split<SH, G, 1>;
    case 2: return k_traverse_split<SH, G, 2>;
    case 4: return k_traverse_split<SH, G, 4>;
    case 8: return k_traverse_split<SH, G, 8>;
    default: return nullptr;
  }
}

template <int SH>
FullKernelPtr split_for_g(int g, int q) {
  return g == 8 ? split_for_q<SH, 8>(q) : g == 4 ? split_for_q<SH, 4>(q) : g == 2 ? split_for_q<SH, 2>(q) : nullptr;
}

}  // namespace

FullKernelPtr split_kernel(int head_levels, int group, int q) {
  switch (head_levels) {
    case 6: return split_for_g<6>(group, q);
    case 7: return split_for_g<7>(group, q);
    default: return nullptr;
  }
}

}  // namespace mlt
