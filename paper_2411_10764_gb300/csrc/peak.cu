// Walk-rate ceiling kernels (measurement only): the full-table walk over
// trees held in shared memory for the whole launch.
#include "peak.cuh"
#include "walk.cuh"

namespace mlt {
namespace walk {

// Walk-rate ceiling of the full-table walk, for measurement: each CTA stages
// its tile (one candidate per thread, as the V pass does) and copies the
// first `resident` trees of the table into shared memory once, then walks
// them `rounds` times with the same node test and layout -- no chunk
// streaming, no barrier between chunks.  out[i] = the fp32 sum, in walk
// order, of the rounds x resident leaves candidate i reaches.
template <int D, int G>
__global__ void __launch_bounds__(kFullMaxTile)
    k_walk_peak(const __grid_constant__ TraverseArgs a, int resident, int rounds, float* out) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int TC = blockDim.x;
  const int tid = threadIdx.x;
  long long tile0;
  int rows_here;
  cta_tile(a, a.n, TC, &tile0, &rows_here);
  if (rows_here <= 0) return;
  float* xs = reinterpret_cast<float*>(smem);
  unsigned char* tbuf = smem + full_smem_tbuf_off(a.F, TC);
  const uint32_t n16 = static_cast<uint32_t>(resident) * (a.tree_bytes / 16u);
  const uint4* src = reinterpret_cast<const uint4*>(a.table);
  uint4* dst = reinterpret_cast<uint4*>(tbuf);
  for (uint32_t i = tid; i < n16; i += blockDim.x) dst[i] = __ldg(src + i);
  const bool nan = __syncthreads_or(stage_row(a, nullptr, xs, nullptr, tile0, rows_here, TC));
  const uint32_t row_bytes = static_cast<uint32_t>(TC) * 4u;
  const unsigned char* xcol = reinterpret_cast<const unsigned char*>(xs) + static_cast<uint32_t>(tid) * 4u;
  float acc = 0.0f;
  for (int r = 0; r < rounds; ++r)
    acc = nan ? walk_chunk<D, G, true, 1>(tbuf, 0, resident, a.tree_bytes, xcol, row_bytes, acc, 0u)
              : walk_chunk<D, G, false, 1>(tbuf, 0, resident, a.tree_bytes, xcol, row_bytes, acc, 0u);
  if (tid < rows_here) out[tile0 + tid] = acc;
}

template <int G>
WalkPeakKernelPtr walk_peak_kernel_for(int d) {
  switch (d) {
    case 1: return k_walk_peak<1, G>;
    case 2: return k_walk_peak<2, G>;
    case 3: return k_walk_peak<3, G>;
    case 4: return k_walk_peak<4, G>;
    case 5: return k_walk_peak<5, G>;
    case 6: return k_walk_peak<6, G>;
    case 7: return k_walk_peak<7, G>;
    case 8: return k_walk_peak<8, G>;
    case 9: return k_walk_peak<9, G>;
    case 10: return k_walk_peak<10, G>;
    default: return nullptr;
  }
}

}  // namespace walk

WalkPeakKernelPtr walk_peak_kernel(int depth, int group) {
  return group == 8   ? walk::walk_peak_kernel_for<8>(depth)
         : group == 4 ? walk::walk_peak_kernel_for<4>(depth)
         : group == 2 ? walk::walk_peak_kernel_for<2>(depth)
                      : nullptr;
}

size_t walk_peak_tree_offset(int F, int TC) { return walk::full_smem_tbuf_off(F, TC); }

}  // namespace mlt
