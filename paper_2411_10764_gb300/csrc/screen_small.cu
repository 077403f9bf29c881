// Single-launch screening of a small batch (ML^2Tuner Sec. 2: V filter, P
// score, keep the (alpha+1)N best; Sec. 3 / Table 3: gbtree ensembles).
//
// For a few thousand candidates the four-kernel sequence (V pass, survivor
// scatter, P pass, top-k) is bound by launch and hand-off latency, not by
// the walk.  Here one kernel does the whole step when both ensembles are
// full tables of the same depth and fit in shared memory together:
//   * every CTA copies the V and P tables into shared memory at once (one
//     bulk copy each, one mbarrier, a bounded wait) while it stages its tile
//     of TC candidates;
//   * Q groups of warps split the trees (each group walks trees q, q + Q,
//     ...), park the leaves, and group 0 adds them in tree order -- the same
//     sequential fp32 sums as the multi-kernel path;
//   * group 0 decides validity against tau, writes pvalid and perf, and
//     appends a rank key per valid candidate;
//   * the last CTA to finish (a ticket, no waiting) selects the top-k: a
//     histogram of the keys over equal-width bins of the batch's score range
//     gives the bin of the k-th key, the keys at or above it are ranked
//     directly (each counts the larger ones), and a bitonic sort of all keys
//     serves when that bin holds too many.
#include <algorithm>

#include "rank.cuh"
#include "walk.cuh"

namespace mlt {
namespace {

using namespace walk;

constexpr int kSmallThreads = 256;
constexpr int kSmallSortMax = kSmallMaxN;  // keys the last CTA can sort (a power of two)
constexpr int kSmallHistBins = 1024;       // equal-width bins over the batch's score range
constexpr unsigned kSmallRankMax = 512;    // rank a collection this small directly

struct SmallArgs {
  const float* feats;  // [n][F]
  int F;
  int n;
  int vec4;
  const unsigned char* v_table;
  const unsigned char* p_table;
  int v_trees;
  int p_trees;
  uint32_t tree_bytes;  // both tables (same depth)
  float tau;
  float* out_pvalid;
  float* out_perf;
  int64_t* out_topk;
  int k;
  unsigned long long* keys;  // [n] scratch
  SelectState* state;        // survivors and ticket (zeroed before the launch)
  unsigned* err;
  int stall_cta;  // failure-detection self-test (-1: none)
  unsigned long long stall_ns;
};

__host__ __device__ constexpr size_t align128(size_t v) { return (v + 127) & ~static_cast<size_t>(127); }

// Shared memory: the two tables, the tile's features [F][TC], parked
// leaves [max(trees)][TC]; the last CTA reuses the start for the selection.
__host__ __device__ inline size_t small_walk_bytes(int F, int TC, int v_trees, int p_trees, uint32_t tb) {
  return align128(static_cast<size_t>(v_trees + p_trees) * tb) + align128(static_cast<size_t>(F) * TC * 4) +
         static_cast<size_t>(v_trees > p_trees ? v_trees : p_trees) * TC * 4;
}
__host__ __device__ constexpr size_t small_select_bytes() {
  return (static_cast<size_t>(kSmallSortMax) + 2) * 8 + kSmallHistBins * 4 + (kSmallRankMax + 2) * 8;
}

// The top-k of the keys[0, m) (m <= kSmallSortMax) by the last CTA.  The
// keys come in with every load of a thread in flight at once.  Up to
// kSmallRankMax keys are ranked directly.  Otherwise a histogram over
// equal-width bins of the score words' range [lo, hi] (bin = (score - lo) x
// scale, non-decreasing in the key, so a better key never lands in a lower
// bin) gives the bin of the kk-th key; the keys in that bin and above are
// collected and ranked, or, if that bin holds too many (equal scores), every
// key is sorted.  Equal-width bins spread a batch's scores over the
// histogram where the top bits of the keys put them in a handful of bins.
__device__ __forceinline__ unsigned small_bin(unsigned long long key, unsigned lo, float scale) {
  const unsigned b = static_cast<unsigned>(static_cast<float>(static_cast<unsigned>(key >> 32) - lo) * scale);
  return b < static_cast<unsigned>(kSmallHistBins) ? b : static_cast<unsigned>(kSmallHistBins) - 1u;
}

__device__ __forceinline__ void select_small(const SmallArgs& s, unsigned m, unsigned char* smem) {
  constexpr int kUnroll = 8;
  const int T = blockDim.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ unsigned warp_sum[kSmallThreads / 32], warp_lo[kSmallThreads / 32], warp_hi[kSmallThreads / 32];
  __shared__ unsigned s_bin;
  unsigned long long* ks = reinterpret_cast<unsigned long long*>(smem);
  unsigned* hist = reinterpret_cast<unsigned*>(ks + kSmallSortMax + 2);
  unsigned long long* cs = reinterpret_cast<unsigned long long*>(hist + kSmallHistBins);
  const unsigned kk = m < static_cast<unsigned>(s.k) ? m : static_cast<unsigned>(s.k);
  unsigned lo = 0xFFFFFFFFu, hi = 0u;
  for (unsigned i0 = 0; i0 < m; i0 += static_cast<unsigned>(T) * kUnroll) {
    unsigned long long v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const unsigned i = i0 + static_cast<unsigned>(u * T + tid);
      v[u] = i < m ? __ldcg(s.keys + i) : 0ull;
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const unsigned i = i0 + static_cast<unsigned>(u * T + tid);
      if (i < m) {
        ks[i] = v[u];
        const unsigned w = static_cast<unsigned>(v[u] >> 32);
        lo = min(lo, w);
        hi = max(hi, w);
      }
    }
  }
  if (kk > 0) {
    if (m <= kSmallRankMax) {
      if (tid == 0 && (m & 1u)) ks[m] = 0ull;
      __syncthreads();
      rank_and_write(ks, m, kk, 0, s.out_topk);
    } else {
      lo = __reduce_min_sync(0xFFFFFFFFu, lo);
      hi = __reduce_max_sync(0xFFFFFFFFu, hi);
      if (lane == 0) {
        warp_lo[warp] = lo;
        warp_hi[warp] = hi;
      }
      for (int b = tid; b < kSmallHistBins; b += T) hist[b] = 0u;
      if (tid == 0) s_bin = 0u;
      __syncthreads();
      for (int w = 0; w < T / 32; ++w) {
        lo = min(lo, warp_lo[w]);
        hi = max(hi, warp_hi[w]);
      }
      const float scale = hi > lo ? (static_cast<float>(kSmallHistBins) - 0.5f) / static_cast<float>(hi - lo) : 0.0f;
      for (unsigned i = tid; i < m; i += T) atomicAdd(&hist[small_bin(ks[i], lo, scale)], 1u);
      __syncthreads();
      // bin of the kk-th largest key: thread t holds the `per` bins just
      // below kSmallHistBins - per t, threads ordered from the top bins down
      constexpr int per = kSmallHistBins / kSmallThreads;
      unsigned h[per];
      unsigned local = 0;
#pragma unroll
      for (int b = 0; b < per; ++b) {
        h[b] = hist[kSmallHistBins - 1 - (tid * per + b)];
        local += h[b];
      }
      unsigned x = local;
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
      }
      if (lane == 31) warp_sum[warp] = x;
      __syncthreads();
      unsigned above = x - local;
      for (int w = 0; w < warp; ++w) above += warp_sum[w];
#pragma unroll
      for (int b = 0; b < per; ++b) {
        if (above < kk && kk <= above + h[b]) s_bin = static_cast<unsigned>(kSmallHistBins - 1 - (tid * per + b));
        above += h[b];
      }
      __syncthreads();
      // the keys of that bin and above (every key better than the kk-th):
      // each thread counts its own, a block scan places them
      const unsigned bin0 = s_bin;
      unsigned mine = 0;
      for (unsigned i = tid; i < m; i += T) mine += small_bin(ks[i], lo, scale) >= bin0 ? 1u : 0u;
      unsigned xs = mine;
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xFFFFFFFFu, xs, o);
        if (lane >= o) xs += y;
      }
      if (lane == 31) warp_sum[warp] = xs;
      __syncthreads();
      unsigned pos = xs - mine, cnt = 0;
      for (int w = 0; w < T / 32; ++w) {
        if (w < warp) pos += warp_sum[w];
        cnt += warp_sum[w];
      }
      if (mine)
        for (unsigned i = tid; i < m; i += T) {
          const unsigned long long key = ks[i];
          if (small_bin(key, lo, scale) >= bin0) {
            if (pos < kSmallRankMax) cs[pos] = key;
            ++pos;
          }
        }
      __syncthreads();
      if (cnt <= kSmallRankMax) {
        if (tid == 0 && (cnt & 1u)) cs[cnt] = 0ull;
        __syncthreads();
        rank_and_write(cs, cnt, kk, 0, s.out_topk);
      } else {
        // a crowded bin: order every key
        int n2 = 2;
        while (n2 < static_cast<int>(m)) n2 <<= 1;
        for (int i = static_cast<int>(m) + tid; i < n2; i += T) ks[i] = 0ull;
        __syncthreads();
        sort_desc(ks, n2);
        for (unsigned r = tid; r < kk; r += T)
          s.out_topk[r] = static_cast<int64_t>(0xFFFFFFFFu - static_cast<uint32_t>(ks[r] & 0xFFFFFFFFull));
      }
    }
  }
  for (int r = static_cast<int>(kk) + tid; r < s.k; r += T) s.out_topk[r] = -1;
}

template <int D, int G, int Q>
__global__ void __launch_bounds__(kSmallThreads) k_screen_small(const __grid_constant__ SmallArgs s) {
  extern __shared__ __align__(128) unsigned char smem[];
  // [0] V table, [2] P table, [1] the self-test's stalled barrier
  __shared__ __align__(8) unsigned long long bars[3];
  __shared__ unsigned s_last;
  const int TC = blockDim.x / Q;
  const int tid = threadIdx.x;
  const int q = tid / TC, c = tid - q * TC;  // q is warp-uniform (TC is a multiple of 32)
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), s.n - tile0));
  const size_t v_bytes = static_cast<size_t>(s.v_trees) * s.tree_bytes;
  const size_t p_bytes = static_cast<size_t>(s.p_trees) * s.tree_bytes;
  unsigned char* vt = smem;
  unsigned char* pt = smem + v_bytes;
  float* xs = reinterpret_cast<float*>(smem + align128(v_bytes + p_bytes));
  float* park = reinterpret_cast<float*>(reinterpret_cast<unsigned char*>(xs) + align128(static_cast<size_t>(s.F) * TC * 4));
  const bool stall = static_cast<int>(blockIdx.x) == s.stall_cta;
  if (tid == 0) {
    for (int b = 0; b < 3; ++b) mbar_init(smem_u32(&bars[b]), 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {  // the tables are static: copy them before waiting on earlier kernels
    // separate barriers, so that the V walk starts while the P table lands
    mbar_expect_tx(smem_u32(&bars[0]), static_cast<uint32_t>(v_bytes));
    bulk_copy_g2s(smem_u32(vt), s.v_table, static_cast<uint32_t>(v_bytes), smem_u32(&bars[0]));
    mbar_expect_tx(smem_u32(&bars[2]), static_cast<uint32_t>(p_bytes));
    bulk_copy_g2s(smem_u32(pt), s.p_table, static_cast<uint32_t>(p_bytes), smem_u32(&bars[2]));
  }
  pdl_wait();
  TraverseArgs ta{};
  ta.feats = s.feats;
  ta.F = s.F;
  ta.vec4 = s.vec4;
  const bool nan = __syncthreads_or(tid < TC && stage_row(ta, nullptr, xs, nullptr, tile0, rows_here, TC));
  const bool ok = stall ? mbar_wait_bounded_ns(smem_u32(&bars[1]), 0u, s.stall_ns)
                        : mbar_wait_bounded(smem_u32(&bars[0]), 0u);
  bool failed = !__syncthreads_and(ok);
  float accv = 0.0f, accp = 0.0f;
  if (!failed) {
    const uint32_t row_bytes = static_cast<uint32_t>(TC) * 4u;
    const unsigned char* xcol = reinterpret_cast<const unsigned char*>(xs) + static_cast<uint32_t>(c) * 4u;
    const uint32_t la = smem_u32(park) + static_cast<uint32_t>(c) * 4u;
    accv = nan ? walk_chunk<D, G, true, Q>(vt, q, s.v_trees, s.tree_bytes, xcol, row_bytes, 0.0f, la)
               : walk_chunk<D, G, false, Q>(vt, q, s.v_trees, s.tree_bytes, xcol, row_bytes, 0.0f, la);
    if (Q > 1) {
      __syncthreads();
      if (q == 0)
        for (int t = 0; t < s.v_trees; ++t) accv += park[t * TC + c];
      __syncthreads();
    }
    failed = !__syncthreads_and(mbar_wait_bounded(smem_u32(&bars[2]), 0u));
    if (!failed) {
      accp = nan ? walk_chunk<D, G, true, Q>(pt, q, s.p_trees, s.tree_bytes, xcol, row_bytes, 0.0f, la)
                 : walk_chunk<D, G, false, Q>(pt, q, s.p_trees, s.tree_bytes, xcol, row_bytes, 0.0f, la);
      if (Q > 1) {
        __syncthreads();
        if (q == 0)
          for (int t = 0; t < s.p_trees; ++t) accp += park[t * TC + c];
      }
    }
  }
  if (failed) {
    if (tid == 0) {
      // both copies land before the CTA's shared memory is released
      mbar_wait_bounded(smem_u32(&bars[0]), 0u);
      mbar_wait_bounded(smem_u32(&bars[2]), 0u);
      atomicOr(s.err, kErrWaitTimeout);
    }
    accv = -INFINITY;  // the tile's bookkeeping still completes, none of it valid
  }
  pdl_trigger();
  if (q == 0) {  // whole warps of group 0
    const bool in = c < rows_here;
    const long long i = tile0 + c;
    const bool valid = in && accv >= s.tau;
    if (in) {
      s.out_pvalid[i] = sigmoid_f(accv);
      s.out_perf[i] = valid ? accp : -INFINITY;
    }
    const unsigned ball = __ballot_sync(0xFFFFFFFFu, valid);
    if (ball) {
      const int lane = tid & 31, leader = __ffs(ball) - 1;
      unsigned pos0 = 0;
      if (lane == leader) pos0 = atomicAdd(&s.state->survivors, static_cast<unsigned>(__popc(ball)));
      pos0 = __shfl_sync(0xFFFFFFFFu, pos0, leader);
      if (valid) s.keys[pos0 + __popc(ball & ((1u << lane) - 1u))] = walk::make_key(accp, static_cast<uint32_t>(i));
    }
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&s.state->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const unsigned m = *reinterpret_cast<volatile unsigned*>(&s.state->survivors);
  select_small(s, m, smem);
  if (tid == 0) s.state->ticket = 0u;
}

using SmallKernelPtr = void (*)(SmallArgs);

template <int Q>
SmallKernelPtr small_for_depth(int d) {
  switch (d) {
    case 1: return k_screen_small<1, 4, Q>;
    case 2: return k_screen_small<2, 4, Q>;
    case 3: return k_screen_small<3, 4, Q>;
    case 4: return k_screen_small<4, 4, Q>;
    case 5: return k_screen_small<5, 4, Q>;
    case 6: return k_screen_small<6, 4, Q>;
    case 7: return k_screen_small<7, 4, Q>;
    case 8: return k_screen_small<8, 4, Q>;
    case 9: return k_screen_small<9, 4, Q>;
    case 10: return k_screen_small<10, 4, Q>;
    default: return nullptr;
  }
}

}  // namespace

SmallPlan plan_small(int F, long long n, const DeviceModel& V, const DeviceModel& P, int sms, int optin) {
  SmallPlan pl{};
  if (n < 1 || n > kSmallMaxN) return pl;
  if (V.kind != kTableFull || P.kind != kTableFull || V.depth != P.depth || V.tree_bytes != P.tree_bytes) return pl;
  if (static_cast<size_t>(V.n_trees + P.n_trees) * V.tree_bytes > kSmallTableBytes) return pl;
  // 256 threads: 32 candidates x 8 tree groups while that spreads the batch
  // over the SMs, else 64 x 4
  const int tc = n <= 32LL * sms ? 32 : 64;
  const size_t smem = std::max(small_walk_bytes(F, tc, V.n_trees, P.n_trees, V.tree_bytes), small_select_bytes());
  if (smem + 1024 > static_cast<size_t>(optin)) return pl;
  pl.threads = tc;
  pl.groups = kSmallThreads / tc;
  pl.smem = smem;
  pl.ctas = static_cast<int>((n + tc - 1) / tc);
  return pl;
}

cudaError_t launch_screen_small(const SmallPlan& pl, const DeviceModel& V, const DeviceModel& P, const float* feats,
                                int F, long long n, float tau, float* out_pvalid, float* out_perf, int64_t* out_topk,
                                int k, const Scratch& sc, int stall_cta, unsigned long long stall_ns,
                                cudaStream_t st) {
  SmallKernelPtr kern = pl.groups == 8 ? small_for_depth<8>(V.depth) : pl.groups == 4 ? small_for_depth<4>(V.depth)
                                                                                         : nullptr;
  if (kern == nullptr) return cudaErrorInvalidValue;
  SmallArgs s{};
  s.feats = feats;
  s.F = F;
  s.n = static_cast<int>(n);
  s.vec4 = ((reinterpret_cast<uintptr_t>(feats) & 15u) == 0 && (F & 3) == 0) ? 1 : 0;
  s.v_table = V.table;
  s.p_table = P.table;
  s.v_trees = V.n_trees;
  s.p_trees = P.n_trees;
  s.tree_bytes = V.tree_bytes;
  s.tau = tau;
  s.out_pvalid = out_pvalid;
  s.out_perf = out_perf;
  s.out_topk = out_topk;
  s.k = k;
  s.keys = sc.keys;
  s.state = sc.state;
  s.err = sc.err;
  s.stall_cta = stall_cta;
  s.stall_ns = stall_ns;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(pl.smem));
  if (e != cudaSuccess) return e;
  e = launch_pdl(kern, dim3(static_cast<unsigned>(pl.ctas)), dim3(kSmallThreads), pl.smem, st, s);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace mlt
