// Split-table walk kernels that build each candidate's features on chip
// from its index (mixed-radix knob decode + feature program, Sec. 2 and
// Appendix A.2) instead of reading a stored feature matrix.
#include "walk.cuh"

namespace mlt {
namespace {

template <int SH, int G, int QS>
__global__ void __launch_bounds__(QS == 8 ? 1024 : 512, 1)
    k_traverse_split_dec(const __grid_constant__ TraverseArgs a, const __grid_constant__ DecodeParams d) {
  walk::traverse_full_body<1, G, QS, false, SH>(a, &d);
}

template <int SH, int G>
FullDecKernelPtr split_dec_for_q(int q) {
  switch (q) {
    case 0: return k_traverse_split_dec<SH, G, 0>;
    case 1: return k_traverse_split_dec<SH, G, 1>;
    case 2: return k_traverse_split_dec<SH, G, 2>;
    case 4: return k_traverse_split_dec<SH, G, 4>;
    case 8: return k_traverse_split_dec<SH, G, 8>;
    default: return nullptr;
  }
}

template <int SH>
FullDecKernelPtr split_dec_for_g(int g, int q) {
  return g == 8 ? split_dec_for_q<SH, 8>(q) : g == 4 ? split_dec_for_q<SH, 4>(q)
         : g == 2 ? split_dec_for_q<SH, 2>(q) : nullptr;
}

}  // namespace

FullDecKernelPtr split_dec_kernel(int head_levels, int group, int q) {
  switch (head_levels) {
    case 6: return split_dec_for_g<6>(group, q);
    case 7: return split_dec_for_g<7>(group, q);
    default: return nullptr;
  }
}

}  // namespace mlt
