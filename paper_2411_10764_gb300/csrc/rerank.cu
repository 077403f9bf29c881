// Model A rerank of the kept candidates.
//
// ML^2Tuner Sec. 2 ("Hidden Feature Extractor & ML Model A"): the explorer
// keeps the (alpha+1)N candidates ranked best by model P, and model A -- a
// regressor over the visible and the compiler's hidden features, deeper
// than P (depth 14, Table 3) -- picks the final N from them.  The batch is
// tiny (tens to a few thousand candidates) and the trees deep, so the walk
// is a chain of dependent loads: one CTA per candidate, its threads walking
// different trees straight from global memory (L1/L2) -- one tree each when
// the batch is small enough to spread over the GPU -- leaves parked in
// shared memory and added by one thread in tree order (the same exact fp32
// sequential sum as the screening walk).  One CTA then sorts the 64-bit keys
// (score, index).
#include <algorithm>

#include "mlt_internal.cuh"

namespace mlt {
namespace {

constexpr int kTreeChunk = 1024;  // leaves parked before summing
constexpr int kSelectThreads = 1024;

__device__ __forceinline__ uint32_t go_right_nan(float x, uint32_t thr_bits, uint32_t meta) {
  uint32_t right = x >= __uint_as_float(thr_bits) ? 1u : 0u;
  if ((x != x) && !(meta & kMetaDefaultLeft)) right = 1u;
  return right;
}

// One tree of a full table, read from global memory (FullLayout).
__device__ float leaf_full(const unsigned char* tree, int D, const float* x) {
  const FullLayout L = full_layout(D);
  uint32_t j = 0;
  for (int l = 0; l < D; ++l) {
    uint32_t thr, meta;
    if (l < static_cast<int>(L.top)) {
      const uint2 r = __ldg(reinterpret_cast<const uint2*>(tree) + j);
      thr = r.x;
      meta = r.y;
    } else {
      const uint32_t m = __ldg(reinterpret_cast<const unsigned short*>(tree + L.off_meta) + (j - L.n_top));
      meta = (m & kMeta16Feature) | ((m & kMeta16Left) ? kMetaDefaultLeft : 0u);
      thr = __ldg(reinterpret_cast<const uint32_t*>(tree + L.off_thr) + (j - L.n_top));
    }
    const float xv = __ldg(x + (meta & ~kMetaDefaultLeft));
    j = 2u * j + 1u + go_right_nan(xv, thr, meta);
  }
  return __ldg(reinterpret_cast<const float*>(tree + L.off_leaf) + (j - L.n_inner));
}

// One tree of a compact table (breadth-first records).
__device__ float leaf_compact(const uint2* tree, const float* x) {
  uint32_t j = 0;
  for (int s = 0; s <= kMaxDepth; ++s) {
    const uint2 r = __ldg(tree + j);
    if (r.y & kMetaLeaf) return __uint_as_float(r.x);
    const float xv = __ldg(x + (r.y & kCompactFeatureMask));
    j = ((r.y >> kCompactChildShift) & kCompactChildMask) + go_right_nan(xv, r.x, r.y);
  }
  return 0.0f;  // unreachable for a validated table
}

struct RerankArgs {
  const float* feats;
  int F;
  long long n;
  const int64_t* cand;
  int m;
  const unsigned char* table;
  int kind;
  int n_trees;
  int depth;
  uint32_t tree_bytes;
  float* out_score;
  unsigned long long* keys;
  unsigned* err;
};

__global__ void __launch_bounds__(1024) k_rerank_walk(const __grid_constant__ RerankArgs a) {
  __shared__ float parked[kTreeChunk];
  pdl_wait();
  const int i = blockIdx.x;  // one candidate per CTA
  const long long c = a.cand[i];
  if (c < 0 || c >= a.n) {
    if (threadIdx.x == 0) {
      a.out_score[i] = -INFINITY;
      a.keys[i] = 0ull;  // sorts below every real key
      if (c >= a.n) atomicOr(a.err, kErrBadIndex);
    }
    return;  // whole CTA
  }
  const float* x = a.feats + c * a.F;
  const uint32_t* offs = reinterpret_cast<const uint32_t*>(a.table);
  const uint2* recs = reinterpret_cast<const uint2*>(a.table + ((static_cast<size_t>(a.n_trees) * 4 + 15) & ~15ull));
  float acc = 0.0f;
  for (int base = 0; base < a.n_trees; base += kTreeChunk) {
    const int nt = min(kTreeChunk, a.n_trees - base);
    for (int t = threadIdx.x; t < nt; t += blockDim.x) {
      const int tree = base + t;
      parked[t] = a.kind == kTableFull ? leaf_full(a.table + static_cast<size_t>(tree) * a.tree_bytes, a.depth, x)
                                       : leaf_compact(recs + __ldg(offs + tree), x);
    }
    __syncthreads();
    if (threadIdx.x == 0)
      for (int t = 0; t < nt; ++t) acc += parked[t];  // tree order
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    a.out_score[i] = acc;
    const uint32_t u = __float_as_uint(acc == 0.0f ? 0.0f : acc);
    const uint32_t mono = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    a.keys[i] = (static_cast<unsigned long long>(mono) << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(c));
  }
}

__global__ void __launch_bounds__(kSelectThreads)
    k_rerank_select(const unsigned long long* keys, int m, int m2, int n_final, int64_t* out) {
  extern __shared__ __align__(16) unsigned long long sk[];
  pdl_wait();
  const int tid = threadIdx.x, T = blockDim.x;
  for (int i = tid; i < m2; i += T) sk[i] = i < m ? keys[i] : 0ull;
  __syncthreads();
  for (int size = 2; size <= m2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = tid; i < (m2 >> 1); i += T) {
        const int lo = (i / stride) * 2 * stride + (i % stride);
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const unsigned long long x = sk[lo], y = sk[hi];
        if ((x < y) == desc) {
          sk[lo] = y;
          sk[hi] = x;
        }
      }
      __syncthreads();
    }
  }
  for (int r = tid; r < n_final; r += T) {
    const unsigned long long key = r < m2 ? sk[r] : 0ull;
    out[r] = key == 0ull ? -1 : static_cast<int64_t>(0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull));
  }
}

}  // namespace

cudaError_t launch_rerank(const DeviceModel& A, const float* feats, int F, long long n, const int64_t* cand, int m,
                          int n_final, float* out_score, int64_t* out_final, unsigned long long* keys,
                          unsigned* err, cudaStream_t st) {
  if (m > 0) {
    RerankArgs a{};
    a.feats = feats;
    a.F = F;
    a.n = n;
    a.cand = cand;
    a.m = m;
    a.table = A.table;
    a.kind = A.kind;
    a.n_trees = A.n_trees;
    a.depth = A.depth;
    a.tree_bytes = A.tree_bytes;
    a.out_score = out_score;
    a.keys = keys;
    a.err = err;
    // threads per candidate: one per tree (a multiple of 32, at most 1,024),
    // fewer when the batch would hold more than 2,048 threads per SM
    int sms = 0, dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long fill = std::max(32LL, static_cast<long long>(sms > 0 ? sms : 1) * 2048 / m / 32 * 32);
    const int threads = static_cast<int>(std::min<long long>({(A.n_trees + 31) / 32 * 32, 1024LL, fill}));
    cudaError_t e = launch_pdl(k_rerank_walk, dim3(static_cast<unsigned>(m)), dim3(threads), 0, st, a);
    if (e != cudaSuccess) return e;
  }
  int m2 = 1;
  while (m2 < m) m2 <<= 1;
  const size_t smem = static_cast<size_t>(m2) * 8;
  cudaError_t e = cudaFuncSetAttribute(k_rerank_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  return launch_pdl(k_rerank_select, dim3(1), dim3(kSelectThreads), smem, st,
                    static_cast<const unsigned long long*>(keys), m, m2, n_final, out_final);
}

}  // namespace mlt
