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
// largest keys" is exactly "k best by (score desc, position asc)"; it also
// counts the keys' top 12 bits in a histogram.  One top-k kernel then finds
// the histogram bucket holding the k-th key, collects every key in that
// bucket or above (a few thousand for the workloads here), and the last CTA
// to finish (ticket counter, no waiting) sorts them in shared memory.  If
// ties crowd more keys into the collection than shared memory holds, that
// CTA first narrows them with an exact most-significant-digit radix select.
#include "mlt_internal.cuh"

namespace mlt {
namespace {

constexpr int kTopkThreads = 512;
constexpr int kSortMin = 8192;  // sort buffer entries (at least pow2(k))

__global__ void __launch_bounds__(256)
    k_scatter(const uint32_t* masks, const uint32_t* offsets, uint32_t* rows, long long n, const StreamState* ss) {
  __shared__ unsigned wc[32];
  pdl_wait();
  pdl_trigger();
  if (ss && *reinterpret_cast<volatile const unsigned*>(&ss->done)) return;
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

// Bitonic sort of sk[0, n2) in descending order (n2 a power of two).
__device__ void sort_desc(unsigned long long* sk, int n2) {
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

__global__ void __launch_bounds__(kTopkThreads)
    k_topk(const unsigned long long* keys, unsigned long long* cand, SelectState* st, int k, int cap,
           long long base, int64_t* out, unsigned* err, const unsigned* count) {
  extern __shared__ __align__(16) unsigned long long sk[];  // cap entries
  __shared__ unsigned warp_sum[kTopkThreads / 32];
  __shared__ unsigned s_bin, s_last, s_digit, s_rem, s_h, s_cnt;
  __shared__ unsigned h256[256];
  pdl_wait();
  const int T = blockDim.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned S = count ? *count : st->survivors;
  const unsigned kk = S < static_cast<unsigned>(k) ? S : static_cast<unsigned>(k);

  // 1. bucket of the kk-th largest key.  Thread t holds the 8 bins
  //    [4096-8(t+1), 4096-8t) in registers; threads are ordered from the top
  //    bins down, so an exclusive scan over threads counts the keys above.
  constexpr int per = kTopBins / kTopkThreads;  // 8
  static_assert(per == 8, "two uint4 loads per thread");
  const uint4* h4 = reinterpret_cast<const uint4*>(st->hist + (kTopBins - per * (tid + 1)));
  const uint4 lo4 = __ldcg(h4), hi4 = __ldcg(h4 + 1);
  const unsigned hb[per] = {hi4.w, hi4.z, hi4.y, hi4.x, lo4.w, lo4.z, lo4.y, lo4.x};  // descending bins
  unsigned local = 0;
#pragma unroll
  for (int q = 0; q < per; ++q) local += hb[q];
  unsigned x = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sum[warp] = x;
  if (tid == 0) s_bin = kTopBins;  // nothing to select unless found
  __syncthreads();
  unsigned above = x - local;
  for (int w = 0; w < warp; ++w) above += warp_sum[w];
#pragma unroll
  for (int q = 0; q < per; ++q) {
    if (kk > 0 && above < kk && kk <= above + hb[q]) s_bin = static_cast<unsigned>(kTopBins - 1 - (tid * per + q));
    above += hb[q];
  }
  __syncthreads();
  const unsigned long long bin = s_bin;

  // 2. collect every key in that bucket or above (warp-aggregated appends)
  for (long long i0 = static_cast<long long>(blockIdx.x) * T; i0 < S; i0 += static_cast<long long>(gridDim.x) * T) {
    const long long i = i0 + tid;
    unsigned long long key = 0;
    bool take = false;
    if (i < S) {
      key = keys[i];
      take = (key >> (64 - kTopBits)) >= bin;
    }
    const unsigned ball = __ballot_sync(0xFFFFFFFFu, take);
    if (ball) {
      const int leader = __ffs(ball) - 1;
      unsigned pos0 = 0;
      if (lane == leader) pos0 = atomicAdd(&st->n_cand, static_cast<unsigned>(__popc(ball)));
      pos0 = __shfl_sync(0xFFFFFFFFu, pos0, leader);
      if (take) cand[pos0 + __popc(ball & ((1u << lane) - 1u))] = key;
    }
  }

  // 3. the last CTA to finish selects and sorts
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&st->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const unsigned m = *reinterpret_cast<volatile unsigned*>(&st->n_cand);
  if (tid == 0) st->v_ticket = 0u;  // in case a V pass ended early
  int n2 = 1;
  while (n2 < static_cast<int>(kk)) n2 <<= 1;
  if (m <= static_cast<unsigned>(cap)) {
    // every collected key fits: sort them all, keep the first kk
    int m2 = 1;
    while (m2 < static_cast<int>(m)) m2 <<= 1;
    for (int i = tid; i < m2; i += T) sk[i] = i < static_cast<int>(m) ? __ldcg(cand + i) : 0ull;
    __syncthreads();
    sort_desc(sk, m2);
  } else {
    // heavy ties: exact radix select of the kk-th key among the collected
    // keys (8-bit digits from the top), then gather the kk keys above it
    unsigned long long prefix = 0, mask = 0;
    unsigned rem = kk;
    for (int shift = 56; shift >= 0; shift -= 8) {
      for (int i = tid; i < 256; i += T) h256[i] = 0u;
      __syncthreads();
      for (unsigned i = tid; i < m; i += T) {
        const unsigned long long key = __ldcg(cand + i);
        if ((key & mask) == prefix) atomicAdd(&h256[(key >> shift) & 0xFFull], 1u);
      }
      __syncthreads();
      if (tid == 0) {
        unsigned cum = 0;
        for (int d = 255; d >= 0; --d) {
          const unsigned h = h256[d];
          if (cum + h >= rem) {
            s_digit = static_cast<unsigned>(d);
            s_rem = rem - cum;
            s_h = h;
            break;
          }
          cum += h;
        }
      }
      __syncthreads();
      prefix |= static_cast<unsigned long long>(s_digit) << shift;
      mask |= 0xFFull << shift;
      rem = s_rem;
      const bool finished = s_h == rem;
      __syncthreads();
      if (finished) break;
    }
    if (tid == 0) s_cnt = 0u;
    __syncthreads();
    for (unsigned i = tid; i < m; i += T) {
      const unsigned long long key = __ldcg(cand + i);
      if ((key & mask) >= prefix) {
        const unsigned p = atomicAdd(&s_cnt, 1u);
        if (p < kk)
          sk[p] = key;
        else
          atomicOr(err, kErrSelect);
      }
    }
    __syncthreads();
    for (int i = static_cast<int>(kk) + tid; i < n2; i += T) sk[i] = 0ull;
    __syncthreads();
    sort_desc(sk, n2);
  }
  for (int r = tid; r < k; r += T) {
    if (r < static_cast<int>(kk)) {
      const uint32_t pos = 0xFFFFFFFFu - static_cast<uint32_t>(sk[r] & 0xFFFFFFFFull);
      out[r] = base + static_cast<long long>(pos);
    } else {
      out[r] = -1;
    }
  }
}

}  // namespace

cudaError_t launch_compact(const Scratch& s, long long n, int tile, long long n_tiles, const StreamState* ss,
                           cudaStream_t st) {
  if (n_tiles <= 0) {
    // no V pass ran: start the selection state from zero survivors
    return cudaMemsetAsync(s.state, 0, sizeof(SelectState), st);
  }
  return launch_pdl(k_scatter, dim3(static_cast<unsigned>(n_tiles)), dim3(tile), 0, st, s.masks,
                    static_cast<const uint32_t*>(s.tile_offsets), s.rows, n, ss);
}

namespace {

// After a batch: add its survivors and candidates to the running counts and
// raise `done` once the target is reached.
__global__ void k_accumulate(StreamState* ss, const SelectState* st, long long n_batch, unsigned target) {
  pdl_wait();
  if (threadIdx.x != 0 || ss->done) return;
  ss->total += st->survivors;
  ss->consumed += static_cast<unsigned long long>(n_batch);
  ss->batches += 1u;
  if (ss->total >= target) ss->done = 1u;
}

__global__ void k_stream_stats(const StreamState* ss, int64_t* out) {
  pdl_wait();
  if (threadIdx.x == 0) {
    out[0] = static_cast<int64_t>(ss->consumed);
    out[1] = static_cast<int64_t>(ss->total);
    out[2] = static_cast<int64_t>(ss->batches);
  }
}

}  // namespace

cudaError_t launch_accumulate(StreamState* ss, const SelectState* st_, long long n_batch, unsigned target,
                              cudaStream_t st) {
  return launch_pdl(k_accumulate, dim3(1), dim3(32), 0, st, ss, st_, n_batch, target);
}

cudaError_t launch_stream_stats(const StreamState* ss, int64_t* out_stats, cudaStream_t st) {
  return launch_pdl(k_stream_stats, dim3(1), dim3(32), 0, st, ss, out_stats);
}

cudaError_t launch_topk(const Scratch& s, long long n, int k, long long index_base, int64_t* out_topk, int sms,
                        const unsigned* count, cudaStream_t st) {
  int cap = kSortMin;
  while (cap < k) cap <<= 1;
  const size_t smem = static_cast<size_t>(cap) * 8;
  cudaError_t e = cudaFuncSetAttribute(k_topk, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  long long g = (n + 1023) / 1024;  // about one pass of the collection loop per warp
  if (g < 1) g = 1;
  if (g > 4LL * sms) g = 4LL * sms;
  return launch_pdl(k_topk, dim3(static_cast<unsigned>(g)), dim3(kTopkThreads), smem, st,
                    static_cast<const unsigned long long*>(s.keys), s.cand, s.state, k, cap, index_base, out_topk,
                    s.err, count);
}

}  // namespace mlt
