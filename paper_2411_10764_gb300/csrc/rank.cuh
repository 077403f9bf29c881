// Ordering of a small set of unique 64-bit rank keys inside one CTA (the
// top-k selection's last step): a bitonic sort, and rank counting (each key
// counts the larger ones), which writes the candidate indices of the kk best
// in order.  Keys: high word = order-preserving image of the P score, low
// word = ~position (see the screening kernels), so a larger key is a better
// candidate (score descending, position ascending).
#pragma once

#include "mlt_internal.cuh"

namespace mlt {

// Bitonic sort of sk[0, n2) in descending order (n2 a power of two).
__device__ __forceinline__ void sort_desc(unsigned long long* sk, int n2) {
  const int tid = threadIdx.x, T = blockDim.x;
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = tid; i < (n2 >> 1); i += T) {
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
}

// Rank of every key among ks[0, m) (keys unique), by counting the larger
// ones; the key of rank r < kk goes to out[r].  p threads share a key (a
// power of two up to 32, as many as the block holds) and add their partial
// counts with shuffles: no barrier, cheaper than a bitonic sort for a few
// hundred keys.  ks[m] must be readable (0 when m is odd: below any key).
__device__ __forceinline__ void rank_and_write(const unsigned long long* ks, unsigned m, unsigned kk, long long base,
                               int64_t* out) {
  const ulonglong2* pairs = reinterpret_cast<const ulonglong2*>(ks);
  const unsigned n_pairs = (m + 1u) >> 1;
  unsigned p = 1;
  while (p < 32u && 2u * p * m <= blockDim.x) p <<= 1;
  if (p == 1) {  // one thread per key: a plain loop the compiler unrolls
    for (unsigned i = threadIdx.x; i < m; i += blockDim.x) {
      const unsigned long long key = ks[i];
      unsigned r = 0;
      for (unsigned j = 0; j < n_pairs; ++j) {
        const ulonglong2 q = pairs[j];
        r += (q.x > key) + (q.y > key);
      }
      if (r < kk) {
        const uint32_t pos = 0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull);
        out[r] = base + static_cast<long long>(pos);
      }
    }
    return;
  }
  const unsigned span = m * p;
  for (unsigned t0 = 0; t0 < span; t0 += blockDim.x) {  // the same trip count in every thread
    const unsigned t = t0 + threadIdx.x;
    const unsigned i = t / p, part = t % p;
    unsigned long long key = 0;
    unsigned r = 0;
    if (t < span) {
      key = ks[i];
      for (unsigned j = part; j < n_pairs; j += p) {
        const ulonglong2 q = pairs[j];
        r += (q.x > key) + (q.y > key);
      }
    }
    for (unsigned o = 1; o < p; o <<= 1) r += __shfl_xor_sync(0xFFFFFFFFu, r, o);
    if (t < span && part == 0 && r < kk) {
      const uint32_t pos = 0xFFFFFFFFu - static_cast<uint32_t>(key & 0xFFFFFFFFull);
      out[r] = base + static_cast<long long>(pos);
    }
  }
}

}  // namespace mlt
