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
// bucket or above (a few hundred to a few thousand for the workloads here),
// and the last CTA to finish (ticket counter, no waiting) orders them.  Up to
// 512 collected keys are ranked directly (each key counts the larger ones);
// a larger collection is first narrowed to exactly the k best with an exact
// most-significant-digit radix select (8-bit digits below the bucket's bits,
// counted in shared memory), whose keys are then ranked the same way (k <=
// 512) or sorted (bitonic).
#include "mlt_internal.cuh"
#include "rank.cuh"

namespace mlt {
namespace {

constexpr int kTopkThreads = 512;
constexpr int kSortMin = 8192;  // collected keys held in shared memory
constexpr unsigned kRankMax = 512;    // order by rank counting up to this many keys
constexpr unsigned kDirectMax = 512;  // rank a collection this small without narrowing it

__global__ void __launch_bounds__(kFullMaxTile)
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

__global__ void __launch_bounds__(kTopkThreads)
    k_topk(const unsigned long long* keys, unsigned long long* cand, SelectState* st, int k, int n2k,
           long long base, int64_t* out, unsigned* err, const unsigned* count) {
  // sk[0, kSortMin): the collected keys when they fit; sk[kSortMin, +n2k):
  // the kk selected keys (n2k = pow2 >= k, at least 2)
  extern __shared__ __align__(16) unsigned long long sk[];
  __shared__ unsigned warp_sum[kTopkThreads / 32];
  __shared__ unsigned s_bin, s_above, s_hbin, s_last, s_digit, s_rem, s_h, s_cnt;
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
    if (kk > 0 && above < kk && kk <= above + hb[q]) {
      s_bin = static_cast<unsigned>(kTopBins - 1 - (tid * per + q));
      s_above = above;
      s_hbin = hb[q];
    }
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

  // 3. the last CTA to finish narrows the collection to exactly the kk best
  //    keys (8-bit digits below the bucket's 12 bits, counted in shared
  //    memory) and orders them
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&st->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const unsigned m = *reinterpret_cast<volatile unsigned*>(&st->n_cand);
  if (tid == 0) st->v_ticket = 0u;  // in case a V pass ended early
  unsigned long long* out_keys = sk + kSortMin;
  if (kk > 0) {
    const bool in_smem = m <= static_cast<unsigned>(kSortMin);
    if (in_smem)
      for (unsigned i = tid; i < m; i += T) sk[i] = __ldcg(cand + i);
    if (m < kk && tid == 0) atomicOr(err, kErrSelect);  // the histogram promised kk
    if (m <= kDirectMax) {
      // a small collection: rank every collected key directly
      if (tid == 0 && (m & 1u)) sk[m] = 0ull;
      __syncthreads();
      rank_and_write(sk, m, kk, base, out);
      for (int r = static_cast<int>(kk) + tid; r < k; r += T) out[r] = -1;
      return;
    }
    auto key_at = [&](unsigned i) { return in_smem ? sk[i] : __ldcg(cand + i); };
    unsigned long long mask = ~0ull << (64 - kTopBits);
    unsigned long long prefix = bin << (64 - kTopBits);
    unsigned rem = kk - s_above;  // keys of the boundary bucket still wanted
    bool finished = s_hbin == rem;
    __syncthreads();
    for (int hi = 64 - kTopBits; hi > 0 && !finished; hi -= 8) {
      const int shift = hi > 8 ? hi - 8 : 0;
      const unsigned long long dmask = (1ull << (hi - shift)) - 1ull;
      if (tid < 256) h256[tid] = 0u;
      __syncthreads();
      for (unsigned i = tid; i < m; i += T) {
        const unsigned long long key = key_at(i);
        if ((key & mask) == prefix) atomicAdd(&h256[(key >> shift) & dmask], 1u);
      }
      __syncthreads();
      // digit of the rem-th key: scan the 256 counts from the top digit down
      unsigned h = 0, incl = 0;
      if (tid < 256) {
        h = h256[255 - tid];
        incl = h;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
          if (lane >= o) incl += y;
        }
        if (lane == 31) warp_sum[warp] = incl;
      }
      __syncthreads();
      if (tid < 256) {
        unsigned ab = incl - h;
        for (int w = 0; w < warp; ++w) ab += warp_sum[w];
        if (ab < rem && rem <= ab + h) {
          s_digit = static_cast<unsigned>(255 - tid);
          s_rem = rem - ab;
          s_h = h;
        }
      }
      __syncthreads();
      prefix |= static_cast<unsigned long long>(s_digit) << shift;
      mask |= dmask << shift;
      rem = s_rem;
      finished = s_h == rem;
      __syncthreads();  // s_* and h256 are rewritten by the next digit
    }
    if (tid == 0) s_cnt = 0u;
    __syncthreads();
    for (unsigned i = tid; i < m; i += T) {
      const unsigned long long key = key_at(i);
      if ((key & mask) >= prefix) {
        const unsigned p = atomicAdd(&s_cnt, 1u);
        if (p < kk)
          out_keys[p] = key;
        else
          atomicOr(err, kErrSelect);
      }
    }
    if (tid == 0 && (kk & 1u)) out_keys[kk] = 0ull;  // pad for the pairwise rank loop (kk odd < n2k)
    __syncthreads();
    if (kk <= kRankMax) {
      rank_and_write(out_keys, kk, kk, base, out);
    } else {
      int n2 = 1;
      while (n2 < static_cast<int>(kk)) n2 <<= 1;
      for (int i = static_cast<int>(kk) + tid; i < n2; i += T) out_keys[i] = 0ull;
      __syncthreads();
      sort_desc(out_keys, n2);
      for (int r = tid; r < static_cast<int>(kk); r += T) {
        const uint32_t pos = 0xFFFFFFFFu - static_cast<uint32_t>(out_keys[r] & 0xFFFFFFFFull);
        out[r] = base + static_cast<long long>(pos);
      }
    }
  }
  for (int r = static_cast<int>(kk) + tid; r < k; r += T) out[r] = -1;
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

namespace {

constexpr int kMergeThreads = 256;
constexpr int kMergeTile = 1024;  // pairs staged in shared memory per pass

// Order-preserving unsigned image of a score (-0 folded onto +0), the high
// word of the screening's rank keys.
__device__ __forceinline__ uint32_t mono_score(float s) {
  const uint32_t u = __float_as_uint(s == 0.0f ? 0.0f : s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Rank of every pair (score, global index) among the m pairs by (score
// descending, index ascending), counted as the number of better pairs
// (indices are unique, so ranks are too); pair i of rank r < k goes to
// out[r].  Pairs with a negative index are empty slots: never ranked,
// never counted.
__global__ void __launch_bounds__(kMergeThreads)
    k_merge_rank(const float* scores, const int64_t* idx, long long m, int k, int64_t* out) {
  __shared__ uint32_t s_key[kMergeTile];
  __shared__ long long s_idx[kMergeTile];
  const long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const bool mine = i < m && idx[i] >= 0;
  const uint32_t key = mine ? mono_score(scores[i]) : 0u;
  const long long id = mine ? static_cast<long long>(idx[i]) : 0;
  long long rank = 0;
  for (long long j0 = 0; j0 < m; j0 += kMergeTile) {
    const int len = static_cast<int>(min(static_cast<long long>(kMergeTile), m - j0));
    __syncthreads();
    for (int t = threadIdx.x; t < len; t += blockDim.x) {
      const long long jj = idx[j0 + t];
      s_key[t] = jj >= 0 ? mono_score(scores[j0 + t]) : 0u;
      s_idx[t] = jj;  // negative: an empty slot
    }
    __syncthreads();
    if (mine)
      for (int t = 0; t < len; ++t) {
        const uint32_t kj = s_key[t];
        const long long ij = s_idx[t];
        rank += (ij >= 0) & ((kj > key) | ((kj == key) & (ij < id)));
      }
  }
  if (mine && rank < k) out[rank] = id;
}

}  // namespace

cudaError_t launch_merge_topk(const float* scores, const int64_t* idx, long long m, int k, int64_t* out,
                              cudaStream_t st) {
  // every slot starts empty (-1: all bits set)
  cudaError_t e = cudaMemsetAsync(out, 0xFF, sizeof(int64_t) * static_cast<size_t>(k), st);
  if (e != cudaSuccess || m <= 0) return e;
  const long long blocks = (m + kMergeThreads - 1) / kMergeThreads;
  k_merge_rank<<<static_cast<unsigned>(blocks), kMergeThreads, 0, st>>>(scores, idx, m, k, out);
  return cudaGetLastError();
}

cudaError_t launch_topk(const Scratch& s, long long n, int k, long long index_base, int64_t* out_topk, int sms,
                        const unsigned* count, cudaStream_t st) {
  int n2k = 2;
  while (n2k < k) n2k <<= 1;
  const size_t smem = static_cast<size_t>(kSortMin + n2k) * 8;
  cudaError_t e = cudaFuncSetAttribute(k_topk, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  long long g = (n + 1023) / 1024;  // about one pass of the collection loop per warp
  if (g < 1) g = 1;
  if (g > 4LL * sms) g = 4LL * sms;
  return launch_pdl(k_topk, dim3(static_cast<unsigned>(g)), dim3(kTopkThreads), smem, st,
                    static_cast<const unsigned long long*>(s.keys), s.cand, s.state, k, n2k, index_base, out_topk,
                    s.err, count);
}

}  // namespace mlt
