// Tree-walk kernels that build each candidate's features on chip from its
// index (mixed-radix knob decode + feature program) instead of reading a
// stored feature matrix, and the materialising decoder of mlt_decode_knobs.
// ML^2Tuner Sec. 2: the explorer enumerates the search space of
// configurations; Appendix A.2: the knobs are tiling sizes and virtual-thread
// counts; Table 5: derived (hidden) features.
#include <algorithm>

#include "walk.cuh"

namespace mlt {
namespace {

using namespace walk;

using CompactDecKernel = void (*)(TraverseArgs, DecodeParams);

CompactDecKernel compact_dec_kernel(int group, int lanes) {
  if (group == 8) {
    switch (lanes) {
      case 1: return k_traverse_compact_dec<8, 1>;
      case 2: return k_traverse_compact_dec<8, 2>;
      case 4: return k_traverse_compact_dec<8, 4>;
      case 8: return k_traverse_compact_dec<8, 8>;
    }
  } else if (group == 4) {
    switch (lanes) {
      case 1: return k_traverse_compact_dec<4, 1>;
      case 2: return k_traverse_compact_dec<4, 2>;
      case 4: return k_traverse_compact_dec<4, 4>;
      case 8: return k_traverse_compact_dec<4, 8>;
    }
  }
  return nullptr;
}

// One thread per candidate: decode into a shared-memory column (stride
// TC + 1, so that both the column writes and the row reads below hit 32
// different banks), then write the rows out coalesced.
__global__ void __launch_bounds__(256)
    k_decode_rows(const __grid_constant__ DecodeParams d, long long n, uint8_t* out_knobs, float* out_feats) {
  extern __shared__ __align__(128) unsigned char smem[];
  float* xs = reinterpret_cast<float*>(smem);
  const int TC = blockDim.x, tid = threadIdx.x, F = d.F;
  const int stride = TC + 1;
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), n - tile0));
  if (tid < rows_here) {
    const long long idx = d.first_index + tile0 + tid;
    decode_column(d, idx, xs, stride, tid);
    if (out_knobs != nullptr) {
      int digit[kMaxKnobs];
      knob_digits(d, idx, digit);
      for (int j = 0; j < d.n_knobs; ++j) out_knobs[(tile0 + tid) * d.n_knobs + j] = static_cast<uint8_t>(digit[j]);
    }
  }
  __syncthreads();
  if (out_feats != nullptr) {
    // element v = r * F + f of the tile's rows, v = tid, tid + TC, ...:
    // (r, f) advance by (TC / F, TC % F) with a carry, no division per step
    const int dr = TC / F, df = TC - dr * F;
    int r = tid / F, f = tid - r * F;
    float* dst = out_feats + tile0 * F;
    for (int v = tid; v < rows_here * F; v += TC) {
      dst[v] = xs[f * stride + r];
      r += dr;
      f += df;
      if (f >= F) {
        f -= F;
        ++r;
      }
    }
  }
}

}  // namespace

FullDecKernelPtr full_dec_kernel_q1(int depth, int group) { return full_dec_kernel_q<1>(depth, group); }

FullDecKernelPtr full_dec_kernel(int depth, int group, int q) {
  switch (q) {
    case 0: return full_dec_kernel_sf(depth, group);
    case 1: return full_dec_kernel_q1(depth, group);
    case 2: return full_dec_kernel_q2(depth, group);
    case 4: return full_dec_kernel_q4(depth, group);
    default: return nullptr;
  }
}

cudaError_t launch_traverse_dec(const DeviceModel& m, const TraverseArgs& args, const DecodeParams& dec,
                                const ScreenShape& shape, long long n_tiles, cudaStream_t st) {
  if (n_tiles <= 0) return cudaSuccess;
  // full-table P pass: whole waves of CTAs, the survivors split evenly over
  // them on the device (CTAs without rows exit at once)
  TraverseArgs a = args;
  long long ctas = n_tiles;
  if (m.kind == kTableHalf) return cudaErrorInvalidValue;  // half tables need stored features
  if (args.p_pass && (m.kind == kTableFull || m.kind == kTableSplit) && shape.p_grid > 0) {
    a.p_wave = shape.p_grid;
    ctas = (n_tiles + shape.p_grid - 1) / shape.p_grid * shape.p_grid;
  }
  const dim3 grid(static_cast<unsigned>(ctas));
  if (m.kind == kTableFull || m.kind == kTableSplit) {
    const int q = shape.sync_free ? 0 : shape.lanes;
    FullDecKernelPtr k = m.kind == kTableSplit ? split_dec_kernel(m.head_levels, shape.group, q)
                                               : full_dec_kernel(m.depth, shape.group, q);
    if (k == nullptr) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(shape.smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(k, grid, dim3(shape.threads * shape.lanes), shape.smem, st, a, dec);
    if (e != cudaSuccess) return e;
  } else {
    CompactDecKernel k = compact_dec_kernel(shape.group, shape.lanes);
    if (k == nullptr) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(shape.smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(k, grid, dim3(shape.threads * shape.lanes), shape.smem, st, a, dec);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_decode_rows(const DecodeParams& dec, long long n, uint8_t* out_knobs, float* out_feats,
                               cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  int tc = 256;
  while (tc > 32 && static_cast<size_t>(dec.F) * (tc + 1) * 4 > 200 * 1024) tc >>= 1;
  const size_t smem = static_cast<size_t>(dec.F) * (tc + 1) * 4;
  cudaError_t e = cudaFuncSetAttribute(k_decode_rows, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long tiles = (n + tc - 1) / tc;
  k_decode_rows<<<static_cast<unsigned>(tiles), tc, smem, st>>>(dec, n, out_knobs, out_feats);
  return cudaGetLastError();
}

}  // namespace mlt
