// Tree-ensemble traversal kernels for batched candidate screening on GB300.
//
// ML^2Tuner (arXiv 2411.10764) Sec. 2: the configuration explorer scores
// candidates with model V (validity) and model P (performance); Sec. 3 /
// Table 3: both are XGBoost gbtree ensembles, so a prediction is the sum
// over trees of the leaf each tree routes the feature vector to.
//
// Layout on chip (one CTA = one tile of candidates, one thread per
// candidate):
//   * the tile's features sit in shared memory transposed, [F][TC+1] fp32:
//     thread c reads x[f] at f*(TC+1)+c, so a warp reading 32 different
//     features of its 32 candidates still hits 32 different banks;
//   * full tables: trees stream through shared memory in chunks with
//     cp.async.bulk (TMA bulk copies) completing on mbarriers, all warps of
//     the CTA walking the same chunk; a thread walks G trees at once for
//     instruction-level parallelism and adds their leaves in tree order, so
//     the fp32 sum is exactly sequential over trees from 0.0f;
//   * compact tables (deep, unbalanced trees): nodes are read from global
//     memory through L1 (they do not fit a shared-memory chunk).
#include <cmath>

#include "mlt_internal.cuh"

namespace mlt {
namespace {

__host__ __device__ constexpr size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// ---------------------------------------------------------------------------
// mbarrier / bulk-copy helpers (inline PTX, sm_90+)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_copy_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for an mbarrier phase, giving up after kWaitLimitNs.
__device__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > kWaitLimitNs) return false;
  }
}

// ---------------------------------------------------------------------------
// Small math helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float sigmoid_f(float m) {
  if (m >= 0.0f) return 1.0f / (1.0f + expf(-m));
  const float e = expf(m);
  return e / (1.0f + e);
}

// 64-bit rank key: larger key = better candidate.  High word: the score
// mapped to an order-preserving unsigned integer (-0 folded onto +0); low
// word: ~position, so equal scores rank the smaller position first.
__device__ __forceinline__ unsigned long long make_key(float s, uint32_t pos) {
  const uint32_t u = __float_as_uint(s == 0.0f ? 0.0f : s);
  const uint32_t mono = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (static_cast<unsigned long long>(mono) << 32) | (0xFFFFFFFFu - pos);
}

// Exact floor(log2 a) for a positive normal float, 0 otherwise.
__device__ __forceinline__ float ilog2_exact(float a) {
  const uint32_t u = __float_as_uint(a);
  const uint32_t e = (u >> 23) & 0xFFu;
  if ((u & 0x80000000u) || e == 0u || e == 0xFFu) return 0.0f;
  return static_cast<float>(static_cast<int>(e) - 127);
}

// ---------------------------------------------------------------------------
// Feature staging: fill xs[f*ROW + c] for the tile's candidates
// ---------------------------------------------------------------------------

// One decoded candidate -> column c of the tile (mixed-radix digits, knob 0
// least significant; then the feature program, one rounded op each).
__device__ bool decode_column(const DecodeParams& d, long long idx, float* xs, int ROW, int c) {
  float kv[kMaxKnobs];
  long long rem = idx;
  for (int j = 0; j < d.n_knobs; ++j) {
    const long long r = d.radix[j];
    const long long q = rem / r;
    const int digit = static_cast<int>(rem - q * r);
    rem = q;
    kv[j] = d.opts[d.opt_off[j] + digit];
  }
  bool nan = false;
  const int nk = d.n_knobs;
  for (int f = 0; f < d.F; ++f) {
    const int sa = d.a[f], sb = d.b[f];
    const float cf = d.c[f];
    const float A = sa < 0 ? cf : (sa < nk ? kv[sa] : xs[(sa - nk) * ROW + c]);
    const float B = sb < 0 ? cf : (sb < nk ? kv[sb] : xs[(sb - nk) * ROW + c]);
    float x;
    switch (d.op[f]) {
      case 0: x = A; break;
      case 1: x = ilog2_exact(A); break;
      case 2: x = __fadd_rn(A, B); break;
      case 3: x = __fsub_rn(A, B); break;
      case 4: x = __fmul_rn(A, B); break;
      case 5: x = __fdiv_rn(A, B); break;
      case 6: x = ceilf(__fdiv_rn(A, B)); break;
      case 7: x = __fsub_rn(A, __fmul_rn(B, floorf(__fdiv_rn(A, B)))); break;
      case 8: x = (B < A) ? B : A; break;
      case 9: x = (B > A) ? B : A; break;
      case 10: x = (A > B) ? 1.0f : 0.0f; break;
      default: x = (A == B) ? 1.0f : 0.0f; break;
    }
    nan |= (x != x);
    xs[f * ROW + c] = x;
  }
  return nan;
}

// Stage the tile; returns whether this thread saw a NaN.  `rowidx` holds
// the survivor positions of the tile in the P pass.
__device__ bool stage_tile(const TraverseArgs& a, const DecodeParams* dec, float* xs,
                           const uint32_t* rowidx, long long tile0, int rows_here, int TC) {
  const int F = a.F;
  const int ROW = TC + 1;
  const int tid = threadIdx.x;
  bool nan = false;
  if (dec != nullptr) {
    if (tid < rows_here) {
      const long long pos = a.p_pass ? static_cast<long long>(rowidx[tid]) : tile0 + tid;
      nan = decode_column(*dec, dec->first_index + pos, xs, ROW, tid);
    } else {
      for (int f = 0; f < F; ++f) xs[f * ROW + tid] = 0.0f;
    }
    return nan;
  }
  if (a.vec4) {
    const int F4 = F >> 2;
    const int nvec = rows_here * F4;
    constexpr int U = 4;
    for (int v0 = tid; v0 < nvec; v0 += TC * U) {
      float4 val[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * TC;
        if (v < nvec) {
          const int r = v / F4;
          const int q = v - r * F4;
          const long long row = a.p_pass ? static_cast<long long>(rowidx[r]) : tile0 + r;
          val[u] = __ldg(reinterpret_cast<const float4*>(a.feats + row * F) + q);
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * TC;
        if (v < nvec) {
          const int r = v / F4;
          const int f = (v - r * F4) << 2;
          xs[(f + 0) * ROW + r] = val[u].x;
          xs[(f + 1) * ROW + r] = val[u].y;
          xs[(f + 2) * ROW + r] = val[u].z;
          xs[(f + 3) * ROW + r] = val[u].w;
          nan |= (val[u].x != val[u].x) | (val[u].y != val[u].y) | (val[u].z != val[u].z) |
                 (val[u].w != val[u].w);
        }
      }
    }
  } else {
    const int nel = rows_here * F;
    for (int v = tid; v < nel; v += TC) {
      const int r = v / F;
      const int f = v - r * F;
      const long long row = a.p_pass ? static_cast<long long>(rowidx[r]) : tile0 + r;
      const float x = __ldg(a.feats + row * F + f);
      xs[f * ROW + r] = x;
      nan |= (x != x);
    }
  }
  // zero the columns past the tile's last candidate
  const int pad = TC - rows_here;
  for (int v = tid; v < pad * F; v += TC) {
    const int f = v / pad;
    const int r = rows_here + (v - f * pad);
    xs[f * ROW + r] = 0.0f;
  }
  return nan;
}

// ---------------------------------------------------------------------------
// Epilogues
// ---------------------------------------------------------------------------
__device__ void finish_tile(const TraverseArgs& a, const uint32_t* rowidx, long long tile0,
                            int rows_here, long long count, float acc) {
  const int tid = threadIdx.x;
  const bool in = tid < rows_here;
  if (a.p_pass) {
    if (in) {
      const uint32_t pos = rowidx[tid];
      a.out_perf[pos] = acc;
      a.keys[tile0 + tid] = make_key(acc, pos);
    }
    return;
  }
  __shared__ unsigned warp_count[32];
  const long long i = tile0 + tid;
  const bool valid = in && (acc >= a.tau);
  if (in) {
    a.out_pvalid[i] = sigmoid_f(acc);
    if (!valid) a.out_perf[i] = -INFINITY;
  }
  const unsigned ball = __ballot_sync(0xFFFFFFFFu, valid);
  const int warp = tid >> 5;
  if ((tid & 31) == 0) {
    if (tile0 + warp * 32 < count) a.masks[(tile0 >> 5) + warp] = ball;
    warp_count[warp] = __popc(ball);
  }
  __syncthreads();
  if (tid == 0) {
    unsigned s = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += warp_count[w];
    a.tile_counts[blockIdx.x] = s;
  }
}

// ---------------------------------------------------------------------------
// Full-table walk of one chunk of trees
// ---------------------------------------------------------------------------
template <int D, int G, bool NANP>
__device__ __forceinline__ float walk_chunk(const unsigned char* tb, int nt, uint32_t tree_bytes,
                                            const unsigned char* xb, uint32_t row_bytes,
                                            uint32_t xoff, float acc) {
  constexpr uint32_t I = (1u << D) - 1u;
  int t = 0;
  for (; t + G <= nt; t += G) {
    const unsigned char* base[G];
    uint32_t j[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      base[g] = tb + static_cast<uint32_t>(t + g) * tree_bytes;
      j[g] = 0;
    }
#pragma unroll
    for (int l = 0; l < D; ++l) {
      uint2 rec[G];
#pragma unroll
      for (int g = 0; g < G; ++g) rec[g] = *reinterpret_cast<const uint2*>(base[g] + j[g] * 8u);
      float x[G];
#pragma unroll
      for (int g = 0; g < G; ++g)
        x[g] = *reinterpret_cast<const float*>(xb + (rec[g].y * row_bytes + xoff));
#pragma unroll
      for (int g = 0; g < G; ++g) {
        uint32_t right = x[g] >= __uint_as_float(rec[g].x) ? 1u : 0u;
        if (NANP && (x[g] != x[g]) && !(rec[g].y >> 31)) right = 1u;
        j[g] = 2u * j[g] + 1u + right;
      }
    }
#pragma unroll
    for (int g = 0; g < G; ++g)
      acc += *reinterpret_cast<const float*>(base[g] + I * 8u + (j[g] - I) * 4u);
  }
  for (; t < nt; ++t) {
    const unsigned char* base = tb + static_cast<uint32_t>(t) * tree_bytes;
    uint32_t j = 0;
#pragma unroll
    for (int l = 0; l < D; ++l) {
      const uint2 rec = *reinterpret_cast<const uint2*>(base + j * 8u);
      const float x = *reinterpret_cast<const float*>(xb + (rec.y * row_bytes + xoff));
      uint32_t right = x >= __uint_as_float(rec.x) ? 1u : 0u;
      if (NANP && (x != x) && !(rec.y >> 31)) right = 1u;
      j = 2u * j + 1u + right;
    }
    acc += *reinterpret_cast<const float*>(base + I * 8u + (j - I) * 4u);
  }
  return acc;
}

template <int D, int G>
__device__ __forceinline__ void traverse_full_body(const TraverseArgs& a, const DecodeParams* dec) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int TC = blockDim.x;
  const int tid = threadIdx.x;
  const int ROW = TC + 1;
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  const long long count = a.p_pass ? static_cast<long long>(a.state->survivors) : a.n;
  if (tile0 >= count) return;  // whole CTA, before any copy is issued
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), count - tile0));

  float* xs = reinterpret_cast<float*>(smem);
  size_t off = align_up(static_cast<size_t>(a.F) * ROW * 4, 128);
  uint32_t* rowidx = reinterpret_cast<uint32_t*>(smem + off);
  off += align_up(static_cast<size_t>(TC) * 4, 128);
  unsigned char* tbuf = smem + off;
  const uint32_t chunk_bytes = static_cast<uint32_t>(a.chunk_trees) * a.tree_bytes;
  off += static_cast<size_t>(a.nbuf) * chunk_bytes;
  unsigned long long* bars = reinterpret_cast<unsigned long long*>(smem + align_up(off, 16));
  const int n_chunks = (a.n_trees + a.chunk_trees - 1) / a.chunk_trees;

  if (tid == 0) {
    for (int b = 0; b < a.nbuf; ++b) mbar_init(smem_u32(&bars[b]), 1);
    fence_mbar_init();
  }
  __syncthreads();
  auto issue = [&](int c, int b) {
    const int first = c * a.chunk_trees;
    const int nt = min(a.chunk_trees, a.n_trees - first);
    const uint32_t bytes = static_cast<uint32_t>(nt) * a.tree_bytes;
    const uint32_t bar = smem_u32(&bars[b]);
    mbar_expect_tx(bar, bytes);
    bulk_copy_g2s(smem_u32(tbuf + static_cast<size_t>(b) * chunk_bytes),
                  a.table + static_cast<size_t>(first) * a.tree_bytes, bytes, bar);
  };
  if (tid == 0)
    for (int c = 0; c < a.nbuf && c < n_chunks; ++c) issue(c, c);

  if (a.p_pass) {
    if (tid < rows_here) rowidx[tid] = a.rows[tile0 + tid];
    __syncthreads();
  }
  const bool nan = __syncthreads_or(stage_tile(a, dec, xs, rowidx, tile0, rows_here, TC));

  float acc = 0.0f;
  const uint32_t row_bytes = static_cast<uint32_t>(ROW) * 4u;  // 4 * odd: bit 31 of meta drops
  const uint32_t xoff = static_cast<uint32_t>(tid) * 4u;
  const unsigned char* xb = smem;
  for (int c = 0; c < n_chunks; ++c) {
    const int b = c % a.nbuf;
    const bool ok = mbar_wait_bounded(smem_u32(&bars[b]), static_cast<uint32_t>(c / a.nbuf) & 1u);
    if (!__syncthreads_and(ok)) {
      if (tid == 0) {
        // let every copy still in flight land before the CTA's shared memory
        // is released, then report
        for (int cc = c + 1; cc < n_chunks && cc < c + a.nbuf; ++cc)
          mbar_wait_bounded(smem_u32(&bars[cc % a.nbuf]), static_cast<uint32_t>(cc / a.nbuf) & 1u);
        mbar_wait_bounded(smem_u32(&bars[b]), static_cast<uint32_t>(c / a.nbuf) & 1u);
        atomicOr(a.err, kErrWaitTimeout);
      }
      return;
    }
    const unsigned char* tb = tbuf + static_cast<size_t>(b) * chunk_bytes;
    const int nt = min(a.chunk_trees, a.n_trees - c * a.chunk_trees);
    acc = nan ? walk_chunk<D, G, true>(tb, nt, a.tree_bytes, xb, row_bytes, xoff, acc)
              : walk_chunk<D, G, false>(tb, nt, a.tree_bytes, xb, row_bytes, xoff, acc);
    __syncthreads();
    if (tid == 0 && c + a.nbuf < n_chunks) issue(c + a.nbuf, b);
  }
  finish_tile(a, rowidx, tile0, rows_here, count, acc);
}

template <int D, int G>
__global__ void __launch_bounds__(256) k_traverse_full(const __grid_constant__ TraverseArgs a) {
  traverse_full_body<D, G>(a, nullptr);
}

template <int D, int G>
__global__ void __launch_bounds__(256)
    k_traverse_full_dec(const __grid_constant__ TraverseArgs a, const __grid_constant__ DecodeParams d) {
  traverse_full_body<D, G>(a, &d);
}

// ---------------------------------------------------------------------------
// Compact-table walk (nodes from global memory)
// ---------------------------------------------------------------------------
template <int G>
__device__ __forceinline__ void traverse_compact_body(const TraverseArgs& a, const DecodeParams* dec) {
  extern __shared__ __align__(128) unsigned char smem[];
  const int TC = blockDim.x;
  const int tid = threadIdx.x;
  const int ROW = TC + 1;
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  const long long count = a.p_pass ? static_cast<long long>(a.state->survivors) : a.n;
  if (tile0 >= count) return;
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), count - tile0));

  float* xs = reinterpret_cast<float*>(smem);
  const size_t off = align_up(static_cast<size_t>(a.F) * ROW * 4, 128);
  uint32_t* rowidx = reinterpret_cast<uint32_t*>(smem + off);
  if (a.p_pass) {
    if (tid < rows_here) rowidx[tid] = a.rows[tile0 + tid];
    __syncthreads();
  }
  const bool nan = __syncthreads_or(stage_tile(a, dec, xs, rowidx, tile0, rows_here, TC));
  (void)nan;  // the compact walk always honours missing values

  const uint32_t* offs = reinterpret_cast<const uint32_t*>(a.table);
  const uint2* recs =
      reinterpret_cast<const uint2*>(a.table + align_up(static_cast<size_t>(a.n_trees) * 4, 16));
  float acc = 0.0f;
  const int steps = a.max_depth + 1;
  int t = 0;
  for (; t < a.n_trees; t += G) {
    const uint2* tr[G];
    uint32_t j[G];
    float leaf[G];
    bool live[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      live[g] = (t + g) < a.n_trees;
      tr[g] = recs + (live[g] ? __ldg(offs + t + g) : 0u);
      j[g] = 0;
      leaf[g] = 0.0f;
    }
    for (int s = 0; s < steps; ++s) {
#pragma unroll
      for (int g = 0; g < G; ++g) {
        if (!live[g]) continue;
        const uint2 r = __ldg(tr[g] + j[g]);
        if (r.y & kMetaLeaf) {
          leaf[g] = __uint_as_float(r.x);
          live[g] = false;
        } else {
          const float x = xs[(r.y & 0xFFFFu) * ROW + tid];
          uint32_t right = x >= __uint_as_float(r.x) ? 1u : 0u;
          if ((x != x) && !(r.y & kMetaDefaultLeft)) right = 1u;
          j[g] = ((r.y >> 16) & 0x3FFFu) + right;
        }
      }
    }
#pragma unroll
    for (int g = 0; g < G; ++g)
      if (t + g < a.n_trees) acc += leaf[g];
  }
  finish_tile(a, rowidx, tile0, rows_here, count, acc);
}

template <int G>
__global__ void __launch_bounds__(256) k_traverse_compact(const __grid_constant__ TraverseArgs a) {
  traverse_compact_body<G>(a, nullptr);
}

template <int G>
__global__ void __launch_bounds__(256)
    k_traverse_compact_dec(const __grid_constant__ TraverseArgs a, const __grid_constant__ DecodeParams d) {
  traverse_compact_body<G>(a, &d);
}

// ---------------------------------------------------------------------------
// Materialising decoder (mlt_decode_knobs)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
    k_decode_rows(const __grid_constant__ DecodeParams d, long long n, uint8_t* out_knobs, float* out_feats) {
  extern __shared__ __align__(128) unsigned char smem[];
  float* xs = reinterpret_cast<float*>(smem);
  const int TC = blockDim.x, ROW = TC + 1, tid = threadIdx.x, F = d.F;
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), n - tile0));
  if (tid < rows_here) {
    const long long idx = d.first_index + tile0 + tid;
    decode_column(d, idx, xs, ROW, tid);
    if (out_knobs != nullptr) {
      long long rem = idx;
      for (int j = 0; j < d.n_knobs; ++j) {
        const long long q = rem / d.radix[j];
        out_knobs[(tile0 + tid) * d.n_knobs + j] = static_cast<uint8_t>(rem - q * d.radix[j]);
        rem = q;
      }
    }
  }
  __syncthreads();
  if (out_feats != nullptr) {
    for (int v = tid; v < rows_here * F; v += TC) {
      const int r = v / F;
      const int f = v - r * F;
      out_feats[(tile0 + r) * F + f] = xs[f * ROW + r];
    }
  }
}

// ---------------------------------------------------------------------------
// Kernel tables
// ---------------------------------------------------------------------------
using FullKernel = void (*)(TraverseArgs);
using FullDecKernel = void (*)(TraverseArgs, DecodeParams);

template <int G>
struct FullTable {
  static FullKernel plain(int d) {
    switch (d) {
      case 1: return k_traverse_full<1, G>;
      case 2: return k_traverse_full<2, G>;
      case 3: return k_traverse_full<3, G>;
      case 4: return k_traverse_full<4, G>;
      case 5: return k_traverse_full<5, G>;
      case 6: return k_traverse_full<6, G>;
      case 7: return k_traverse_full<7, G>;
      case 8: return k_traverse_full<8, G>;
      case 9: return k_traverse_full<9, G>;
      case 10: return k_traverse_full<10, G>;
      default: return nullptr;
    }
  }
  static FullDecKernel dec(int d) {
    switch (d) {
      case 1: return k_traverse_full_dec<1, G>;
      case 2: return k_traverse_full_dec<2, G>;
      case 3: return k_traverse_full_dec<3, G>;
      case 4: return k_traverse_full_dec<4, G>;
      case 5: return k_traverse_full_dec<5, G>;
      case 6: return k_traverse_full_dec<6, G>;
      case 7: return k_traverse_full_dec<7, G>;
      case 8: return k_traverse_full_dec<8, G>;
      case 9: return k_traverse_full_dec<9, G>;
      case 10: return k_traverse_full_dec<10, G>;
      default: return nullptr;
    }
  }
};

constexpr size_t kSmPerSm = 228 * 1024;   // shared memory per SM
constexpr size_t kCtaReserve = 1024;      // reserved per resident CTA

}  // namespace

ScreenShape plan_full(int F, int depth, int n_trees, uint32_t tree_bytes, int optin) {
  (void)depth;
  ScreenShape s{};
  s.threads = 256;
  const size_t feat = align_up(static_cast<size_t>(F) * (s.threads + 1) * 4, 128);
  const size_t fixed = feat + align_up(static_cast<size_t>(s.threads) * 4, 128) + 16 + 8 * 4 + 256;
  // two resident CTAs per SM if a chunk of >= 4 trees still fits twice,
  // otherwise one CTA with the rest of shared memory for tree chunks
  for (int ctas = 2; ctas >= 1; --ctas) {
    size_t budget = kSmPerSm / ctas - kCtaReserve;
    if (budget > static_cast<size_t>(optin)) budget = static_cast<size_t>(optin);
    if (budget <= fixed) continue;
    const size_t trees_fit = (budget - fixed) / tree_bytes;
    const int group = ctas == 2 ? 4 : 8;
    int chunk = static_cast<int>(trees_fit / 2);
    if (chunk > 16) chunk = 16;
    if (chunk > n_trees) chunk = n_trees;
    if (chunk >= group) chunk -= chunk % group;
    if (chunk < 1) continue;
    if (ctas == 2 && chunk < 4 && n_trees >= 4) continue;
    int nbuf = static_cast<int>(trees_fit / static_cast<size_t>(chunk));
    if (nbuf > 3) nbuf = 3;
    if (nbuf < 1) continue;
    s.chunk_trees = chunk;
    s.nbuf = nbuf;
    s.group = chunk >= 8 && ctas == 1 ? 8 : 4;
    s.smem = fixed + static_cast<size_t>(nbuf) * chunk * tree_bytes;
    return s;
  }
  s.threads = 0;  // does not fit
  return s;
}

ScreenShape plan_compact(int F, int optin) {
  ScreenShape best{};
  int best_threads = -1;
  for (int tc : {256, 128, 64, 32}) {
    const size_t smem = align_up(static_cast<size_t>(F) * (tc + 1) * 4, 128) +
                        align_up(static_cast<size_t>(tc) * 4, 128);
    if (smem > static_cast<size_t>(optin)) continue;
    int ctas = static_cast<int>(kSmPerSm / (smem + kCtaReserve));
    if (ctas < 1) continue;
    int resident = ctas * tc;
    if (resident > 2048) resident = 2048;
    if (resident > best_threads) {
      best_threads = resident;
      best.threads = tc;
      best.smem = smem;
    }
  }
  best.group = 4;
  best.chunk_trees = 0;
  best.nbuf = 0;
  return best;
}

cudaError_t launch_traverse(const DeviceModel& m, const TraverseArgs& args, const DecodeParams* dec,
                            const ScreenShape& shape, long long n_tiles, cudaStream_t st) {
  if (n_tiles <= 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>(n_tiles)), block(shape.threads);
  if (m.kind == kTableFull) {
    if (dec == nullptr) {
      FullKernel k = shape.group == 8 ? FullTable<8>::plain(m.depth) : FullTable<4>::plain(m.depth);
      if (k == nullptr) return cudaErrorInvalidValue;
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(shape.smem));
      if (e != cudaSuccess) return e;
      k<<<grid, block, shape.smem, st>>>(args);
    } else {
      FullDecKernel k = shape.group == 8 ? FullTable<8>::dec(m.depth) : FullTable<4>::dec(m.depth);
      if (k == nullptr) return cudaErrorInvalidValue;
      cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(shape.smem));
      if (e != cudaSuccess) return e;
      k<<<grid, block, shape.smem, st>>>(args, *dec);
    }
  } else {
    if (dec == nullptr) {
      cudaError_t e = cudaFuncSetAttribute(k_traverse_compact<4>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(shape.smem));
      if (e != cudaSuccess) return e;
      k_traverse_compact<4><<<grid, block, shape.smem, st>>>(args);
    } else {
      cudaError_t e = cudaFuncSetAttribute(k_traverse_compact_dec<4>,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           static_cast<int>(shape.smem));
      if (e != cudaSuccess) return e;
      k_traverse_compact_dec<4><<<grid, block, shape.smem, st>>>(args, *dec);
    }
  }
  return cudaGetLastError();
}

cudaError_t launch_decode_rows(const DecodeParams& dec, long long n, uint8_t* out_knobs,
                               float* out_feats, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const int tc = 256;
  const size_t smem = static_cast<size_t>(dec.F) * (tc + 1) * 4;
  cudaError_t e = cudaFuncSetAttribute(k_decode_rows, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const long long tiles = (n + tc - 1) / tc;
  k_decode_rows<<<static_cast<unsigned>(tiles), tc, smem, st>>>(dec, n, out_knobs, out_feats);
  return cudaGetLastError();
}

}  // namespace mlt
