// Survivor compaction and deterministic top-k for batched candidate
// screening.
//
// ML^2Tuner Sec. 2: a candidate model V predicts invalid is never profiled,
// and the explorer keeps the (alpha+1)N survivors that model P ranks
// highest.  Here: the V pass leaves one 32-bit ballot per warp and one count
// per tile; an exclusive scan of the tile counts and a scatter turn them
// into the ascending list of survivor positions (stable, no atomics on the
// order).  The P pass leaves one 64-bit key per survivor (score mapped to an
// order-preserving integer, then ~position), so keys are unique and "k
// largest keys" is exactly "k best by (score desc, position asc)".  A
// most-significant-digit radix select (six passes of 11/11/11/11/11/9 bits)
// finds the k-th key without any inter-CTA waiting: the last CTA of each
// pass (ticket counter) picks the digit.  The <= k selected keys are then
// sorted in one CTA (bitonic) and written as indices.
#include "mlt_internal.cuh"

namespace mlt {
namespace {

constexpr int kScanThreads = 1024;
constexpr int kPassThreads = 256;
constexpr int kSortThreads = 1024;

__global__ void __launch_bounds__(kScanThreads)
    k_scan(const uint32_t* counts, uint32_t* offsets, long long n_tiles, SelectState* st, int k) {
  __shared__ unsigned part[kScanThreads];
  const int T = blockDim.x, tid = threadIdx.x;
  const long long per = (n_tiles + T - 1) / T;
  const long long b = tid * per;
  const long long e = min(n_tiles, b + per);
  unsigned s = 0;
  for (long long i = b; i < e; ++i) s += counts[i];
  part[tid] = s;
  __syncthreads();
  for (int off = 1; off < T; off <<= 1) {
    const unsigned v = tid >= off ? part[tid - off] : 0u;
    __syncthreads();
    part[tid] += v;
    __syncthreads();
  }
  unsigned run = part[tid] - s;
  for (long long i = b; i < e; ++i) {
    offsets[i] = run;
    run += counts[i];
  }
  if (tid == T - 1) {
    const unsigned total = part[T - 1];
    st->survivors = total;
    st->k = static_cast<unsigned>(k);
    st->prefix = 0ull;
    st->mask = 0ull;
    st->remaining = total < static_cast<unsigned>(k) ? total : static_cast<unsigned>(k);
    st->done = total <= static_cast<unsigned>(k) ? 1u : 0u;
    st->ticket = 0u;
    st->n_sel = 0u;
  }
  for (int i = tid; i < kRadixBins; i += T) st->hist[i] = 0u;
}

__global__ void __launch_bounds__(256)
    k_scatter(const uint32_t* masks, const uint32_t* offsets, uint32_t* rows, long long n) {
  __shared__ unsigned wc[32];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const long long tile0 = static_cast<long long>(blockIdx.x) * blockDim.x;
  const long long first = tile0 + warp * 32;
  const unsigned m = first < n ? masks[first >> 5] : 0u;
  if (lane == 0) wc[warp] = __popc(m);
  __syncthreads();
  unsigned base = offsets[blockIdx.x];
  for (int w = 0; w < warp; ++w) base += wc[w];
  if ((m >> lane) & 1u) rows[base + __popc(m & ((1u << lane) - 1u))] = static_cast<uint32_t>(first + lane);
}

__device__ __forceinline__ int pass_shift(int pass) { return pass < 5 ? 53 - 11 * pass : 0; }
__device__ __forceinline__ int pass_width(int pass) { return pass < 5 ? 11 : 9; }

__global__ void __launch_bounds__(kPassThreads)
    k_radix_pass(const unsigned long long* keys, SelectState* st, int pass) {
  __shared__ unsigned hist[kRadixBins];
  __shared__ unsigned part[kPassThreads];
  __shared__ unsigned is_last;
  if (st->done) return;  // written by an earlier kernel; uniform
  const int tid = threadIdx.x, T = blockDim.x;
  const unsigned S = st->survivors;
  const int shift = pass_shift(pass), width = pass_width(pass);
  const int nb = 1 << width;
  const unsigned long long dmask = (1ull << width) - 1ull;
  const unsigned long long mask = st->mask, prefix = st->prefix;
  const unsigned rem = st->remaining;  // read before the last CTA rewrites it
  for (int i = tid; i < nb; i += T) hist[i] = 0u;
  __syncthreads();
  for (long long i = static_cast<long long>(blockIdx.x) * T + tid; i < S;
       i += static_cast<long long>(gridDim.x) * T) {
    const unsigned long long key = keys[i];
    if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & dmask], 1u);
  }
  __syncthreads();
  for (int i = tid; i < nb; i += T)
    if (hist[i]) atomicAdd(&st->hist[i], hist[i]);
  __threadfence();
  __syncthreads();
  if (tid == 0) is_last = atomicAdd(&st->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  // Last CTA: pick the digit of the rem-th largest prefix-matching key.
  // Thread t owns reversed positions [t*per, (t+1)*per): digits nb-1-r.
  const int per = nb / T;  // nb is a multiple of T
  unsigned local = 0;
  for (int q = 0; q < per; ++q) {
    const int d = nb - 1 - (tid * per + q);
    const unsigned h = __ldcg(&st->hist[d]);
    hist[d] = h;
    local += h;
  }
  part[tid] = local;
  __syncthreads();
  for (int off = 1; off < T; off <<= 1) {
    const unsigned v = tid >= off ? part[tid - off] : 0u;
    __syncthreads();
    part[tid] += v;
    __syncthreads();
  }
  unsigned above = part[tid] - local;  // keys on digits above this thread's range
  for (int q = 0; q < per; ++q) {
    const int d = nb - 1 - (tid * per + q);
    const unsigned h = hist[d];
    if (above < rem && rem <= above + h) {
      const unsigned left = rem - above;
      st->remaining = left;
      st->prefix = prefix | (static_cast<unsigned long long>(d) << shift);
      st->mask = mask | (dmask << shift);
      st->done = (left == h || pass == kRadixPasses - 1) ? 1u : 0u;
    }
    above += h;
  }
  __syncthreads();
  for (int i = tid; i < kRadixBins; i += T) st->hist[i] = 0u;
  if (tid == 0) st->ticket = 0u;
}

__global__ void __launch_bounds__(256)
    k_gather(const unsigned long long* keys, SelectState* st, unsigned long long* sel, unsigned* err) {
  const unsigned S = st->survivors;
  const unsigned long long mask = st->mask, prefix = st->prefix;
  const unsigned k = st->k;
  for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < S;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const unsigned long long key = keys[i];
    if ((key & mask) >= prefix) {
      const unsigned p = atomicAdd(&st->n_sel, 1u);
      if (p < k)
        sel[p] = key;
      else
        atomicOr(err, kErrSelect);
    }
  }
}

__global__ void __launch_bounds__(kSortThreads)
    k_sort_out(const SelectState* st, const unsigned long long* sel, int k, int n2, long long base,
               int64_t* out) {
  extern __shared__ __align__(16) unsigned long long sk[];
  const int tid = threadIdx.x, T = blockDim.x;
  const unsigned cnt_raw = st->n_sel;
  const int cnt = static_cast<int>(cnt_raw < static_cast<unsigned>(k) ? cnt_raw : static_cast<unsigned>(k));
  for (int i = tid; i < n2; i += T) sk[i] = i < cnt ? sel[i] : 0ull;
  __syncthreads();
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
  for (int r = tid; r < k; r += T) {
    if (r < cnt) {
      const uint32_t pos = 0xFFFFFFFFu - static_cast<uint32_t>(sk[r] & 0xFFFFFFFFull);
      out[r] = base + static_cast<long long>(pos);
    } else {
      out[r] = -1;
    }
  }
}

int pass_grid(long long n) {
  long long g = (n + 4095) / 4096;
  if (g < 1) g = 1;
  if (g > 608) g = 608;
  return static_cast<int>(g);
}

}  // namespace

cudaError_t launch_compact(const Scratch& s, long long n, int tile, long long n_tiles, int k,
                           cudaStream_t st) {
  k_scan<<<1, kScanThreads, 0, st>>>(s.tile_counts, s.tile_offsets, n_tiles, s.state, k);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (n_tiles > 0) k_scatter<<<static_cast<unsigned>(n_tiles), tile, 0, st>>>(s.masks, s.tile_offsets, s.rows, n);
  return cudaGetLastError();
}

cudaError_t launch_topk(const Scratch& s, long long n, int k, long long index_base, int64_t* out_topk,
                        cudaStream_t st) {
  const int g = pass_grid(n);
  for (int p = 0; p < kRadixPasses; ++p) {
    k_radix_pass<<<g, kPassThreads, 0, st>>>(s.keys, s.state, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  k_gather<<<g, 256, 0, st>>>(s.keys, s.state, s.sel, s.err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int n2 = 1;
  while (n2 < k) n2 <<= 1;
  const size_t smem = static_cast<size_t>(n2) * 8;
  e = cudaFuncSetAttribute(k_sort_out, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  k_sort_out<<<1, kSortThreads, smem, st>>>(s.state, s.sel, k, n2, index_base, out_topk);
  return cudaGetLastError();
}

}  // namespace mlt
