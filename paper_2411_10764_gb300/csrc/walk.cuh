// Device code of the tree-ensemble walk (included by traverse.cu and
// traverse_dec.cu, which instantiate the plain and the decoding kernels).
//
// ML^2Tuner (arXiv 2411.10764) Sec. 2: the configuration explorer scores
// candidates with model V (validity) and model P (performance); Sec. 3 /
// Table 3: both are XGBoost gbtree ensembles, so a prediction is the sum
// over trees of the leaf each tree routes the feature vector to.
//
// Layout on chip (one CTA = one tile of TC candidates, one thread each):
//   * the tile's features sit in shared memory transposed, [F][TC] fp32:
//     thread c reads x[f] at f*TC + c, so its bank is c mod 32 whatever f
//     is -- a warp gathering 32 different features of its 32 candidates is
//     conflict-free;
//   * full tables: trees stream through shared memory in chunks with
//     cp.async.bulk (bulk TMA copies) completing on mbarriers, all warps of
//     the CTA walking the same chunk; a thread walks G trees at once for
//     instruction-level parallelism and adds their leaves in tree order, so
//     the fp32 sum is exactly sequential over trees from 0.0f;
//   * compact tables (deep, unbalanced trees): nodes are read from global
//     memory through L1 (they do not fit a shared-memory chunk).
#pragma once

#include <cmath>

#include <cuda_fp16.h>

#include "mlt_internal.cuh"

namespace mlt {
namespace walk {

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

// L2 cache policies for loads: node tables of the deep-tree walk are
// re-read by every tile and should stay in L2 (evict_last); feature rows are
// read once and should leave first (evict_first).
__device__ __forceinline__ unsigned long long policy_evict_last() {
  unsigned long long p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ unsigned long long policy_evict_first() {
  unsigned long long p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint2 ldg_u2_hint(const uint2* ptr, unsigned long long pol) {
  uint2 v;
  asm("ld.global.nc.L2::cache_hint.v2.u32 {%0, %1}, [%2], %3;" : "=r"(v.x), "=r"(v.y) : "l"(ptr), "l"(pol));
  return v;
}
__device__ __forceinline__ float4 ldg_f4_hint(const float4* ptr, unsigned long long pol) {
  float4 v;
  asm("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
      : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
      : "l"(ptr), "l"(pol));
  return v;
}

// Wait for an mbarrier phase, giving up after limit_ns nanoseconds.
__device__ __forceinline__ bool mbar_wait_bounded_ns(uint32_t bar, uint32_t parity, unsigned long long limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = global_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (global_ns() - t0 > limit_ns) return false;
  }
}

// Wait for an mbarrier phase, giving up after kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
  return mbar_wait_bounded_ns(bar, parity, kWaitLimitNs);
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
// Feature staging: thread c fills column c of xs[f*TC + c]
// ---------------------------------------------------------------------------

// One decoded candidate -> column c of the tile (mixed-radix digits, knob 0
// least significant; then the feature program, one rounded op each).
// Mixed-radix digit j of candidate idx for every j (knob 0 least
// significant): 32-bit divisions while the index fits 32 bits (a 64-bit
// division is a long subroutine), 64-bit ones otherwise.
__device__ __forceinline__ void knob_digits(const DecodeParams& d, long long idx, int* digit) {
  if ((static_cast<unsigned long long>(idx) >> 32) == 0) {
    uint32_t rem = static_cast<uint32_t>(idx);
    for (int j = 0; j < d.n_knobs; ++j) {
      const uint32_t r = static_cast<uint32_t>(d.radix[j]);
      const uint32_t q = rem / r;
      digit[j] = static_cast<int>(rem - q * r);
      rem = q;
    }
  } else {
    long long rem = idx;
    for (int j = 0; j < d.n_knobs; ++j) {
      const long long r = d.radix[j];
      const long long q = rem / r;
      digit[j] = static_cast<int>(rem - q * r);
      rem = q;
    }
  }
}

__device__ __forceinline__ bool decode_column(const DecodeParams& d, long long idx, float* xs, int TC,
                                              int c) {
  float kv[kMaxKnobs];
  if ((static_cast<unsigned long long>(idx) >> 32) == 0) {
    uint32_t rem = static_cast<uint32_t>(idx);
    for (int j = 0; j < d.n_knobs; ++j) {
      const uint32_t r = static_cast<uint32_t>(d.radix[j]);
      const uint32_t q = rem / r;
      kv[j] = d.opts[d.opt_off[j] + static_cast<int>(rem - q * r)];
      rem = q;
    }
  } else {
    long long rem = idx;
    for (int j = 0; j < d.n_knobs; ++j) {
      const long long r = d.radix[j];
      const long long q = rem / r;
      kv[j] = d.opts[d.opt_off[j] + static_cast<int>(rem - q * r)];
      rem = q;
    }
  }
  bool nan = false;
  const int nk = d.n_knobs;
  for (int f = 0; f < d.F; ++f) {
    const int sa = d.a[f], sb = d.b[f];
    const float cf = d.c[f];
    const float A = sa < 0 ? cf : (sa < nk ? kv[sa] : xs[(sa - nk) * TC + c]);
    const float B = sb < 0 ? cf : (sb < nk ? kv[sb] : xs[(sb - nk) * TC + c]);
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
    xs[f * TC + c] = x;
  }
  return nan;
}

// Stage this thread's candidate (one row per thread: the 32 lanes of a
// store hit 32 different banks).  Returns whether the row holds a NaN.
__device__ __forceinline__ bool stage_row(const TraverseArgs& a, const DecodeParams* dec, float* xs,
                                          const uint32_t* rowidx, long long tile0, int rows_here,
                                          int TC, bool read_once = false) {
  const int F = a.F;
  const int c = threadIdx.x;
  if (c >= rows_here) {
    for (int f = 0; f < F; ++f) xs[f * TC + c] = 0.0f;
    return false;
  }
  const long long pos = a.p_pass ? static_cast<long long>(rowidx[c]) : tile0 + c;
  if (dec != nullptr)
    return decode_column(*dec, dec->index_list ? dec->index_list[pos] : dec->first_index + pos, xs, TC, c);
  bool nan = false;
  const float* src = a.feats + pos * F;
  if (a.vec4) {
    const float4* s4 = reinterpret_cast<const float4*>(src);
    const int F4 = F >> 2;
    constexpr int U = 8;
    for (int q0 = 0; q0 < F4; q0 += U) {
      float4 v[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (q0 + u < F4) v[u] = read_once ? ldg_f4_hint(s4 + q0 + u, policy_evict_first()) : __ldg(s4 + q0 + u);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (q0 + u < F4) {
          const int f = (q0 + u) << 2;
          xs[(f + 0) * TC + c] = v[u].x;
          xs[(f + 1) * TC + c] = v[u].y;
          xs[(f + 2) * TC + c] = v[u].z;
          xs[(f + 3) * TC + c] = v[u].w;
          nan |= (v[u].x != v[u].x) | (v[u].y != v[u].y) | (v[u].z != v[u].z) | (v[u].w != v[u].w);
        }
      }
    }
  } else {
    for (int f = 0; f < F; ++f) {
      const float x = __ldg(src + f);
      xs[f * TC + c] = x;
      nan |= (x != x);
    }
  }
  return nan;
}

// ---------------------------------------------------------------------------
// Epilogues
// ---------------------------------------------------------------------------

// Exclusive scan of the per-tile survivor counts by one CTA, then the
// survivor total and a fresh selection state for the P pass and top-k.
__device__ __forceinline__ void scan_tiles(const uint32_t* counts, uint32_t* offsets, long long n_tiles,
                                           SelectState* st, bool reset_hist) {
  __shared__ unsigned warp_sum[32];
  __shared__ unsigned carry;
  const int T = blockDim.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = T >> 5;
  if (tid == 0) carry = 0;
  __syncthreads();
  for (long long base = 0; base < n_tiles; base += T) {
    const long long i = base + tid;
    const unsigned v = i < n_tiles ? __ldcg(counts + i) : 0u;
    unsigned x = v;  // inclusive warp scan
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_sum[warp] = x;
    __syncthreads();
    unsigned before = carry;
    for (int w = 0; w < warp; ++w) before += warp_sum[w];
    if (i < n_tiles) offsets[i] = before + x - v;
    __syncthreads();
    if (tid == T - 1) carry = before + x;
    __syncthreads();
  }
  if (tid == 0) {
    st->survivors = carry;
    st->n_cand = 0u;
    st->ticket = 0u;
    st->v_ticket = 0u;
  }
  if (reset_hist)
    for (int i = tid; i < kTopBins; i += T) st->hist[i] = 0u;
  (void)nw;
}
// Threads [0, tc) hold the tile's candidates (tc = candidates per CTA, a
// multiple of 32); every thread of the CTA calls this.
__device__ __forceinline__ void finish_tile(const TraverseArgs& a, const uint32_t* rowidx,
                                            long long tile0, int rows_here, long long count, float acc,
                                            int tc) {
  const int tid = threadIdx.x;
  const bool in = tid < rows_here;
  if (a.p_pass) {
    unsigned bin = 0xFFFFFFFFu;
    if (in) {
      const uint32_t pos = rowidx[tid];
      if (a.out_perf) a.out_perf[pos] = acc;
      // batched accumulation: keys of all batches side by side, positions
      // counted from the call's first candidate
      const long long key_base = a.stream ? static_cast<long long>(a.stream->total) : 0;
      const unsigned long long key = make_key(acc, static_cast<uint32_t>(a.pos_base + pos));
      a.keys[key_base + tile0 + tid] = key;
      bin = static_cast<unsigned>(key >> (64 - kTopBits));
    }
    // one atomic per distinct bucket of the warp
    const unsigned peers = __match_any_sync(0xFFFFFFFFu, bin);
    if (in && (tid & 31) == __ffs(peers) - 1) atomicAdd(&a.hist[bin], static_cast<unsigned>(__popc(peers)));
    return;
  }
  __shared__ unsigned warp_count[32];
  const long long i = tile0 + tid;
  const bool valid = in && (acc >= a.tau);
  if (in) {
    if (a.out_pvalid) a.out_pvalid[i] = sigmoid_f(acc);
    if (!valid && a.out_perf) a.out_perf[i] = -INFINITY;
  }
  const unsigned ball = __ballot_sync(0xFFFFFFFFu, valid);
  const int warp = tid >> 5;
  if ((tid & 31) == 0) {
    if (warp * 32 < tc && tile0 + warp * 32 < count) a.masks[(tile0 >> 5) + warp] = ball;
    warp_count[warp] = __popc(ball);
  }
  __shared__ unsigned is_last;
  __syncthreads();
  if (tid == 0) {
    unsigned s = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += warp_count[w];
    a.tile_counts[blockIdx.x] = s;
    __threadfence();
    is_last = atomicAdd(&a.state_rw->v_ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (is_last) {
    // the last V tile to finish turns the tile counts into offsets and
    // resets the selection state (no CTA waits for another)
    __threadfence();
    // batched accumulation keeps the key histogram of earlier batches
    scan_tiles(a.tile_counts, a.tile_offsets, gridDim.x, a.state_rw, a.stream == nullptr);
  }
}

// ---------------------------------------------------------------------------
// Full-table walk of one chunk of trees
// ---------------------------------------------------------------------------
// 32-bit shared-window loads.  `volatile` keeps them in program order with
// the barriers and mbarrier waits around the walk; the walk below issues the
// G trees' loads of one level back to back, so ordering costs no overlap.
__device__ __forceinline__ uint2 lds_u2(uint32_t a) {
  uint2 v;
  asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
  return v;
}
__device__ __forceinline__ uint4 lds_u4(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
  return v;
}
__device__ __forceinline__ uint32_t lds_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
  return v;
}
__device__ __forceinline__ float lds_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a));
  return v;
}

// Go right?  x >= threshold; a missing x takes the node's default side.
template <bool NANP>
__device__ __forceinline__ uint32_t go_right(float x, uint32_t thr_bits, uint32_t meta) {
  uint32_t right = x >= __uint_as_float(thr_bits) ? 1u : 0u;
  if (NANP && (x != x) && !(meta >> 31)) right = 1u;
  return right;
}

__device__ __forceinline__ void sts_f32(uint32_t a, float v) {
  asm volatile("st.shared.f32 [%0], %1;" ::"r"(a), "f"(v) : "memory");
}

// Walk trees q, q + Q, q + 2Q, ... (< nt) of the chunk at shared address tb;
// xa = shared address of this thread's feature column (feature f at xa + f *
// row_bytes).  Q == 1: the leaves are added to acc in tree order.  Q > 1:
// leaf t is parked at la + t * row_bytes for an in-order sum afterwards.
// The 32-bit product meta * row_bytes drops a 4-byte meta's bit 31 because
// row_bytes is a multiple of 2; a 2-byte meta is masked to its feature.
// Shared-memory loads of the walk as ordinary C++ loads through pointers
// derived from the kernel's shared array (so they compile to shared-memory
// loads the compiler may schedule freely among the G walks); the mbarrier
// waits around the walk carry a memory clobber, so no load moves across
// them.
template <typename T>
__device__ __forceinline__ T ld_sm(const unsigned char* p, uint32_t off) {
  return *reinterpret_cast<const T*>(p + off);
}

// Node j of a full-table tree at level l (a compile-time constant after
// unrolling): threshold bits, the feature's byte offset in the staged tile,
// and the NaN-goes-left flag in bit 31.
template <int D>
struct FullNode {
  uint32_t thr, xoff, left;
};
template <int D>
__device__ __forceinline__ FullNode<D> full_node(const unsigned char* base, int l, uint32_t j, uint32_t row_bytes) {
  constexpr FullLayout L = full_layout(D);
  // byte offsets folded with the heap index of each region's first node
  constexpr uint32_t kThr = L.off_thr - L.n_top * 4u;
  constexpr uint32_t kMeta = L.off_meta - L.n_top * 2u;
  FullNode<D> n;
  if (l < static_cast<int>(L.top)) {
    const uint2 r = ld_sm<uint2>(base, j * 8u);
    n.thr = r.x;
    n.xoff = r.y * row_bytes;
    n.left = r.y;
  } else {
    const uint32_t m = ld_sm<unsigned short>(base, kMeta + j * 2u);
    n.thr = ld_sm<uint32_t>(base, kThr + j * 4u);
    n.xoff = (m & kMeta16Feature) * row_bytes;
    n.left = m << 16;
  }
  return n;
}

template <int D, int G, bool NANP, int Q>
__device__ __forceinline__ float walk_chunk(const unsigned char* tb, int q, int nt, uint32_t tree_bytes,
                                            const unsigned char* xc, uint32_t row_bytes, float acc, uint32_t la) {
  constexpr FullLayout L = full_layout(D);
  constexpr uint32_t kLeaf = L.off_leaf - L.n_inner * 4u;  // leaf of child heap index c at kLeaf + 4c
  int t = q;
  for (; t + (G - 1) * Q < nt; t += G * Q) {
    const unsigned char* base[G];
    uint32_t j[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      base[g] = tb + static_cast<uint32_t>(t + g * Q) * tree_bytes;
      j[g] = 0;
    }
#pragma unroll
    for (int l = 0; l < D; ++l) {
      FullNode<D> n[G];
#pragma unroll
      for (int g = 0; g < G; ++g) n[g] = full_node<D>(base[g], l, j[g], row_bytes);
      float x[G];
#pragma unroll
      for (int g = 0; g < G; ++g) x[g] = ld_sm<float>(xc, n[g].xoff);
#pragma unroll
      for (int g = 0; g < G; ++g) j[g] = 2u * j[g] + 1u + go_right<NANP>(x[g], n[g].thr, n[g].left);
    }
    float lf[G];
#pragma unroll
    for (int g = 0; g < G; ++g) lf[g] = ld_sm<float>(base[g], kLeaf + j[g] * 4u);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if (Q == 1)
        acc += lf[g];
      else
        sts_f32(la + static_cast<uint32_t>(t + g * Q) * row_bytes, lf[g]);
    }
  }
  for (; t < nt; t += Q) {
    const unsigned char* base = tb + static_cast<uint32_t>(t) * tree_bytes;
    uint32_t j = 0;
#pragma unroll
    for (int l = 0; l < D; ++l) {
      const FullNode<D> n = full_node<D>(base, l, j, row_bytes);
      const float x = ld_sm<float>(xc, n.xoff);
      j = 2u * j + 1u + go_right<NANP>(x, n.thr, n.left);
    }
    const float leaf = ld_sm<float>(base, kLeaf + j * 4u);
    if (Q == 1)
      acc += leaf;
    else
      sts_f32(la + static_cast<uint32_t>(t) * row_bytes, leaf);
  }
  return acc;
}

// Shared-memory layout of the full-table kernel (host and device agree):
//   features [F][TC] (xb = 4 bytes each, 2 for half tables); rows [TC] u32;
//   nbuf chunk buffers; with Q > 1 tree groups, two parked-leaf buffers
//   [chunk_trees][TC] fp32; mbarriers.
__host__ __device__ inline size_t full_smem_rows_off(int F, int TC, int xb = 4) {
  return align_up(static_cast<size_t>(F) * TC * xb, 128);
}
__host__ __device__ inline size_t full_smem_tbuf_off(int F, int TC, int xb = 4) {
  return full_smem_rows_off(F, TC, xb) + align_up(static_cast<size_t>(TC) * 4, 128);
}
__host__ __device__ inline size_t full_smem_leaf_off(int F, int TC, int nbuf, uint32_t chunk_bytes, int xb = 4) {
  return align_up(full_smem_tbuf_off(F, TC, xb) + static_cast<size_t>(nbuf) * chunk_bytes, 16);
}
__host__ __device__ inline size_t full_smem_leaf_bytes(int TC, int Q, int chunk_trees) {
  return Q > 1 ? 2 * static_cast<size_t>(chunk_trees) * TC * 4 : 0;
}
__host__ __device__ inline size_t full_smem_bytes(int F, int TC, int nbuf, uint32_t chunk_bytes, int Q,
                                                  int chunk_trees, int xb = 4) {
  return full_smem_leaf_off(F, TC, nbuf, chunk_bytes, xb) + full_smem_leaf_bytes(TC, Q, chunk_trees) + 8 * 4;
}

// ---------------------------------------------------------------------------
// Half-table walk (binary16 thresholds, leaves and staged features)
// ---------------------------------------------------------------------------
// Stage this thread's candidate as binary16 (round to nearest even; NaN
// stays NaN, magnitudes past 65504 become infinities).  Returns whether the
// row holds a NaN.
__device__ __forceinline__ bool stage_row_half(const TraverseArgs& a, unsigned short* xs, const uint32_t* rowidx,
                                               long long tile0, int rows_here, int TC) {
  const int F = a.F;
  const int c = threadIdx.x;
  if (c >= rows_here) {
    for (int f = 0; f < F; ++f) xs[f * TC + c] = 0;
    return false;
  }
  const long long pos = a.p_pass ? static_cast<long long>(rowidx[c]) : tile0 + c;
  const float* src = a.feats + pos * F;
  bool nan = false;
  if (a.vec4) {
    const float4* s4 = reinterpret_cast<const float4*>(src);
    for (int q = 0; q < (F >> 2); ++q) {
      const float4 v = ldg_f4_hint(s4 + q, policy_evict_first());
      const int f = q << 2;
      xs[(f + 0) * TC + c] = __half_as_ushort(__float2half_rn(v.x));
      xs[(f + 1) * TC + c] = __half_as_ushort(__float2half_rn(v.y));
      xs[(f + 2) * TC + c] = __half_as_ushort(__float2half_rn(v.z));
      xs[(f + 3) * TC + c] = __half_as_ushort(__float2half_rn(v.w));
      nan |= (v.x != v.x) | (v.y != v.y) | (v.z != v.z) | (v.w != v.w);
    }
  } else {
    for (int f = 0; f < F; ++f) {
      const float x = __ldg(src + f);
      xs[f * TC + c] = __half_as_ushort(__float2half_rn(x));
      nan |= (x != x);
    }
  }
  return nan;
}

__device__ __forceinline__ unsigned short lds_u16(uint32_t a) {
  unsigned short v;
  asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
  return v;
}

// Go right?  x >= threshold in binary16; a missing x takes the node's
// default side (bit 31 of the node word).
template <bool NANP>
__device__ __forceinline__ uint32_t go_right_half(unsigned short x, uint32_t w) {
  const __half xh = __ushort_as_half(x);
  uint32_t right = __hge(xh, __ushort_as_half(static_cast<unsigned short>(w & 0xFFFFu))) ? 1u : 0u;
  if (NANP && __hisnan(xh) && !(w >> 31)) right = 1u;
  return right;
}

// Walk trees [0, nt) of a half-table chunk at shared address tb; xa = shared
// address of this thread's binary16 feature column (feature f at xa + f *
// row_bytes).  Leaves (binary16, exact in fp32) are added in tree order.
template <int D, int G, bool NANP>
__device__ __forceinline__ float walk_chunk_half(uint32_t tb, int nt, uint32_t tree_bytes, uint32_t xa,
                                                 uint32_t row_bytes, float acc) {
  constexpr HalfLayout L = half_layout(D);
  constexpr uint32_t kLast = L.off_last - L.n_inner * 8u;
  int t = 0;
  for (; t + G <= nt; t += G) {
    uint32_t base[G], j[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      base[g] = tb + static_cast<uint32_t>(t + g) * tree_bytes;
      j[g] = 0;
    }
#pragma unroll
    for (int l = 0; l < D - 1; ++l) {
      uint32_t w[G];
#pragma unroll
      for (int g = 0; g < G; ++g) w[g] = lds_u32(base[g] + j[g] * 4u);
      unsigned short x[G];
#pragma unroll
      for (int g = 0; g < G; ++g)
        x[g] = lds_u16(((w[g] >> kHalfFeatureShift) & kHalfFeatureMask) * row_bytes + xa);
#pragma unroll
      for (int g = 0; g < G; ++g) j[g] = 2u * j[g] + 1u + go_right_half<NANP>(x[g], w[g]);
    }
    uint2 r[G];
#pragma unroll
    for (int g = 0; g < G; ++g) r[g] = lds_u2(base[g] + kLast + j[g] * 8u);
    unsigned short x[G];
#pragma unroll
    for (int g = 0; g < G; ++g) x[g] = lds_u16(((r[g].x >> kHalfFeatureShift) & kHalfFeatureMask) * row_bytes + xa);
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint32_t bits = go_right_half<NANP>(x[g], r[g].x) ? (r[g].y >> 16) : (r[g].y & 0xFFFFu);
      acc += __half2float(__ushort_as_half(static_cast<unsigned short>(bits)));
    }
  }
  for (; t < nt; ++t) {
    const uint32_t base = tb + static_cast<uint32_t>(t) * tree_bytes;
    uint32_t j = 0;
#pragma unroll
    for (int l = 0; l < D - 1; ++l) {
      const uint32_t w = lds_u32(base + j * 4u);
      const unsigned short x = lds_u16(((w >> kHalfFeatureShift) & kHalfFeatureMask) * row_bytes + xa);
      j = 2u * j + 1u + go_right_half<NANP>(x, w);
    }
    const uint2 r = lds_u2(base + kLast + j * 8u);
    const unsigned short x = lds_u16(((r.x >> kHalfFeatureShift) & kHalfFeatureMask) * row_bytes + xa);
    const uint32_t bits = go_right_half<NANP>(x, r.x) ? (r.y >> 16) : (r.y & 0xFFFFu);
    acc += __half2float(__ushort_as_half(static_cast<unsigned short>(bits)));
  }
  return acc;
}

// ---------------------------------------------------------------------------
// Split-table walk (deep trees: a shared-memory head, a global-memory tail)
// ---------------------------------------------------------------------------
// Walk trees q, q + Q, ... (< nt) of a chunk of head blocks at shared
// address tb (head_bytes apart): H levels of 8-byte records and the exit
// record from shared memory, then -- only where the exit is a split node --
// the tail records from global memory (`tails`, kept in L2 with
// evict_last), at most tail_steps of them.  The G walks of a thread issue
// their tail loads together, and a warp stops once all its walks sit on a
// leaf.  Q == 1: leaves added to acc in tree order; Q > 1: leaf t parked at
// la + t * row_bytes for group 0's in-order sum.
// Split-table test: every node sends a missing value right.  A node whose
// missing values go left is stored with its children swapped, bit 31 of its
// meta set and threshold -prev(t) (prev(t) = the float below t): then
// "x < t or x missing" (the old left side, now right) is exactly "-x >= -prev(t)
// or -x missing" -- one sign flip and one unordered compare per visit, no
// missing-value branch.
__device__ __forceinline__ uint32_t go_right_split(float x, uint32_t thr_bits, uint32_t meta) {
  const float xs = __uint_as_float(__float_as_uint(x) ^ (meta & 0x80000000u));
  return !(xs < __uint_as_float(thr_bits)) ? 1u : 0u;
}

// A tail record load that only the live walkers issue (v keeps its value
// where p is false), so the tail loop has no branch per walker.
__device__ __forceinline__ void ldg_u2_hint_if(bool p, const uint2* ptr, unsigned long long pol, uint2& v) {
  asm("{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %3, 0;\n\t"
      "@q ld.global.nc.L2::cache_hint.v2.u32 {%0, %1}, [%2], %4;\n\t}"
      : "+r"(v.x), "+r"(v.y)
      : "l"(ptr), "r"(p ? 1 : 0), "l"(pol));
}

template <int H, int G, int Q>
__device__ __forceinline__ float walk_chunk_split(const unsigned char* tb, int q, int nt, uint32_t head_bytes,
                                                  const unsigned char* xc, uint32_t row_bytes, float acc, uint32_t la,
                                                  const uint2* tails, int tail_steps) {
  const unsigned long long keep = policy_evict_last();
  for (int t = q; t < nt; t += G * Q) {
    const unsigned char* base[G];
    uint32_t j[G];
    bool in[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      in[g] = t + g * Q < nt;
      base[g] = tb + static_cast<uint32_t>(in[g] ? t + g * Q : t) * head_bytes;
      j[g] = 0;
    }
#pragma unroll
    for (int l = 0; l < H; ++l) {
      uint2 r[G];
#pragma unroll
      for (int g = 0; g < G; ++g) r[g] = ld_sm<uint2>(base[g], j[g] * 8u);
      float x[G];
#pragma unroll
      for (int g = 0; g < G; ++g) x[g] = ld_sm<float>(xc, r[g].y * row_bytes);
#pragma unroll
      for (int g = 0; g < G; ++g) j[g] = 2u * j[g] + 1u + go_right_split(x[g], r[g].x, r[g].y);
    }
    // the exit record (level H) and the tree's tail base
    uint2 r[G];
    uint32_t tbase[G];
    bool live[G];
#pragma unroll
    for (int g = 0; g < G; ++g) {
      r[g] = ld_sm<uint2>(base[g], j[g] * 8u);
      tbase[g] = ld_sm<uint32_t>(base[g], head_bytes - 8u);
      live[g] = in[g] && !(r[g].y & kMetaLeaf);
    }
    // every walker computes its next index (a leaf record reads feature 0
    // and child 0); only the live ones load.  The loop runs the table's
    // full tail depth with no warp vote: a vote per step ties the G walkers'
    // load chains together (none could start its next step before all G
    // loads returned), and some lane of a warp nearly always walks to the
    // bottom anyway (workload 5's shape: 6 % faster without the vote)
    for (int s = 0; s < tail_steps; ++s) {
      float x[G];
#pragma unroll
      for (int g = 0; g < G; ++g) x[g] = ld_sm<float>(xc, (r[g].y & kCompactFeatureMask) * row_bytes);
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const uint32_t idx =
            tbase[g] + ((r[g].y >> kCompactChildShift) & kCompactChildMask) + go_right_split(x[g], r[g].x, r[g].y);
        ldg_u2_hint_if(live[g], tails + idx, keep, r[g]);
      }
#pragma unroll
      for (int g = 0; g < G; ++g) live[g] = live[g] && !(r[g].y & kMetaLeaf);
    }
#pragma unroll
    for (int g = 0; g < G; ++g) {
      if (!in[g]) continue;
      const float leaf = __uint_as_float(r[g].x);
      if (Q == 1)
        acc += leaf;
      else
        sts_f32(la + static_cast<uint32_t>(t + g * Q) * row_bytes, leaf);
    }
  }
  return acc;
}

// Even split of `len` items into `parts` contiguous pieces whose sizes
// differ by at most one; piece i starts at split_start(len, parts, i).  The
// survivor count is a 32-bit value, so 32-bit arithmetic suffices (a 64-bit
// division would become a call inside the kernel).
__device__ __forceinline__ uint32_t split_start(uint32_t len, uint32_t parts, uint32_t i) {
  const uint32_t base = len / parts, rem = len % parts;
  return i * base + min(i, rem);
}

// The tile of a CTA.  V pass: candidates [blockIdx.x * TC, +TC).  P pass:
// the S survivors are split evenly into A tiles of at most TC rows, A a
// multiple of `per_wave` (the CTAs one wave holds, a.p_wave) unless S is
// small, then one tile per 32 rows at most -- so every SM gets the same
// share whatever S turns out to be.  CTAs past A have no tile (len 0).
__device__ __forceinline__ void cta_tile(const TraverseArgs& a, long long count, int TC, long long* tile0,
                                         int* len) {
  if (!a.p_pass) {
    *tile0 = static_cast<long long>(blockIdx.x) * TC;
    *len = static_cast<int>(max(0LL, min(static_cast<long long>(TC), count - *tile0)));
    return;
  }
  const uint32_t S = static_cast<uint32_t>(count);
  const uint32_t wave = a.p_wave > 0 ? static_cast<uint32_t>(a.p_wave) : gridDim.x;
  const uint32_t waves = (S + static_cast<uint32_t>(TC) * wave - 1) / (static_cast<uint32_t>(TC) * wave);
  const uint32_t tiles = min(min(waves * wave, (S + 31u) / 32u), gridDim.x);
  if (blockIdx.x >= tiles) {
    *tile0 = count;
    *len = 0;
    return;
  }
  const uint32_t lo = split_start(S, tiles, blockIdx.x);
  *tile0 = lo;
  *len = static_cast<int>(split_start(S, tiles, blockIdx.x + 1) - lo);
}

// Full-table walk of one tile.  The CTA has Q groups of TC threads (TC =
// candidates of the tile, a multiple of 32).  Thread c of group q walks
// trees q, q + Q, ... of every chunk for candidate c; with Q > 1 it parks
// the leaves in shared memory and group 0 adds each chunk's leaves in tree
// order one chunk later (two leaf buffers), so the sum is the same
// sequential fp32 sum as with one walker.  More groups put more warps on a
// small batch; all lanes of a warp still walk the same tree.
// QS = tree groups, or 0 for one group with the barrier-free chunk
// pipeline: each warp counts itself out of a chunk buffer and the last one
// refills it, so warps drift up to nbuf - 1 chunks apart instead of meeting
// at a CTA barrier per chunk.  That wins where one CTA holds the SM; with two
// resident CTAs the barrier version keeps the refills further ahead.
// SH > 0: a split table with SH head levels (tree_bytes = the head block;
// D is unused).
template <int D, int G, int QS, bool H = false, int SH = 0>
__device__ __forceinline__ void traverse_full_body(const TraverseArgs& a, const DecodeParams* dec) {
  constexpr int Q = QS == 0 ? 1 : QS;
  constexpr bool kSyncFree = QS == 0;
  static_assert(!H || Q == 1, "half tables walk with one tree group");
  constexpr int xb = H ? 2 : 4;  // bytes per staged feature
  extern __shared__ __align__(128) unsigned char smem[];
  const int TC = blockDim.x / Q;
  const int tid = threadIdx.x;
  const int q = Q == 1 ? 0 : tid / TC;  // warp-uniform (TC is a multiple of 32)
  const int c = Q == 1 ? tid : tid - q * TC;
  // the P pass needs the survivor count of the kernels before it; the V
  // pass only needs them before it reads the features, unless a batched call
  // must first learn whether an earlier batch already reached its target
  if (a.p_pass || a.stream) pdl_wait();
  if (a.stream && *reinterpret_cast<volatile const unsigned*>(&a.stream->done)) return;
  const long long count = a.p_pass ? static_cast<long long>(a.state->survivors) : a.n;
  long long tile0;
  int rows_here;
  cta_tile(a, count, TC, &tile0, &rows_here);
  if (rows_here <= 0) return;  // whole CTA, before any copy is issued

  float* xs = reinterpret_cast<float*>(smem);
  uint32_t* rowidx = reinterpret_cast<uint32_t*>(smem + full_smem_rows_off(a.F, TC, xb));
  unsigned char* tbuf = smem + full_smem_tbuf_off(a.F, TC, xb);
  const uint32_t chunk_bytes = static_cast<uint32_t>(a.chunk_trees) * a.tree_bytes;
  const size_t leaf_off = full_smem_leaf_off(a.F, TC, a.nbuf, chunk_bytes, xb);
  unsigned long long* bars = reinterpret_cast<unsigned long long*>(
      smem + leaf_off + full_smem_leaf_bytes(TC, Q, a.chunk_trees));
  const int n_chunks = (a.n_trees + a.chunk_trees - 1) / a.chunk_trees;
  // barrier-free pipeline: warps release a chunk buffer by counting
  // themselves out; the last one refills it
  __shared__ unsigned released[4];
  __shared__ int last_issued[4];  // latest chunk copied into each buffer

  // bars[3] is never completed (nbuf <= 3): the self-test's stalled wait
  const bool stall = static_cast<int>(blockIdx.x) == a.stall_cta;
  if (tid == 0) {
    for (int b = 0; b < a.nbuf; ++b) mbar_init(smem_u32(&bars[b]), 1);
    if (stall) mbar_init(smem_u32(&bars[3]), 1);
    for (int b = 0; b < 4; ++b) {
      released[b] = 0u;
      last_issued[b] = b < n_chunks ? b : -1;
    }
    fence_mbar_init();
  }
  __syncthreads();
  auto issue = [&](int ch, int b) {
    const int first = ch * a.chunk_trees;
    const int nt = min(a.chunk_trees, a.n_trees - first);
    const uint32_t bytes = static_cast<uint32_t>(nt) * a.tree_bytes;
    const uint32_t bar = smem_u32(&bars[b]);
    mbar_expect_tx(bar, bytes);
    bulk_copy_g2s(smem_u32(tbuf + static_cast<size_t>(b) * chunk_bytes),
                  a.table + static_cast<size_t>(first) * a.tree_bytes, bytes, bar);
  };
  if (tid == 0)
    for (int ch = 0; ch < a.nbuf && ch < n_chunks; ++ch) issue(ch, ch);  // tables are static

  if (!a.p_pass) pdl_wait();
  if (a.p_pass && tid < rows_here) rowidx[tid] = a.rows[tile0 + tid];
  // group 0 stages one row per thread (a thread reads only its own rowidx
  // entry); every group reads the same feature columns
  bool nan;
  if constexpr (H)
    nan = __syncthreads_or(stage_row_half(a, reinterpret_cast<unsigned short*>(xs), rowidx, tile0, rows_here, TC));
  else
    nan = __syncthreads_or(tid < TC && stage_row(a, dec, xs, rowidx, tile0, rows_here, TC));
  // warps past the tile's rows walk zero features: a branch around their
  // walk measured slower than the idle work (it changes the code of the
  // walk loop)
  const bool live = (c & ~31) < rows_here;

  float acc = 0.0f;
  const uint32_t row_bytes = static_cast<uint32_t>(TC) * xb;
  const uint32_t xa = smem_u32(xs) + static_cast<uint32_t>(c) * xb;
  const unsigned char* xcol = reinterpret_cast<const unsigned char*>(xs) + static_cast<uint32_t>(c) * xb;
  const uint32_t tbuf_a = smem_u32(tbuf);
  // parked leaves: buffer p holds leaf t of candidate c at la[p] + t * row_bytes
  const uint32_t la0 = smem_u32(smem + leaf_off) + static_cast<uint32_t>(c) * 4u;
  const uint32_t la_step = static_cast<uint32_t>(a.chunk_trees) * row_bytes;
  // wait for chunk ch in buffer b (bounded); the self-test's stalled CTA
  // waits for its first chunk on bars[3] instead
  auto chunk_wait = [&](int ch, int b) -> bool {
    if (stall && ch == 0) return mbar_wait_bounded_ns(smem_u32(&bars[3]), 0u, a.stall_ns);
    return mbar_wait_bounded(smem_u32(&bars[b]), static_cast<uint32_t>(ch / a.nbuf) & 1u);
  };
  bool failed = false;
  if constexpr (kSyncFree) {
    const int n_warps = static_cast<int>(blockDim.x >> 5);
    const int lane = tid & 31;
    bool timed_out = false;
    for (int ch = 0; ch < n_chunks; ++ch) {
      const int b = ch % a.nbuf;
      const bool ok = chunk_wait(ch, b);
      if (!__all_sync(0xFFFFFFFFu, ok)) {
        timed_out = true;
        break;
      }
      const uint32_t tb = tbuf_a + static_cast<uint32_t>(b) * chunk_bytes;
      const int nt = min(a.chunk_trees, a.n_trees - ch * a.chunk_trees);
      if constexpr (H)
        acc = nan ? walk_chunk_half<D, G, true>(tb, nt, a.tree_bytes, xa, row_bytes, acc)
                  : walk_chunk_half<D, G, false>(tb, nt, a.tree_bytes, xa, row_bytes, acc);
      else if constexpr (SH > 0)
        acc = walk_chunk_split<SH, G, 1>(tbuf + (tb - tbuf_a), 0, nt, a.tree_bytes, xcol, row_bytes, acc, 0u, a.tail,
                                         a.max_depth - SH);
      else
        acc = nan ? walk_chunk<D, G, true, 1>(tbuf + (tb - tbuf_a), 0, nt, a.tree_bytes, xcol, row_bytes, acc, 0u)
                  : walk_chunk<D, G, false, 1>(tbuf + (tb - tbuf_a), 0, nt, a.tree_bytes, xcol, row_bytes, acc, 0u);
      __syncwarp();
      if (lane == 0 && ch + a.nbuf < n_chunks) {
        __threadfence_block();  // this warp's reads of buffer b are done
        if (atomicAdd(&released[b], 1u) == static_cast<unsigned>(n_warps - 1)) {
          released[b] = 0u;
          last_issued[b] = ch + a.nbuf;
          __threadfence_block();
          issue(ch + a.nbuf, b);  // the last warp out refills it
        }
      }
    }
    if (__syncthreads_or(timed_out)) {
      if (tid == 0) {
        // the copy last issued into each buffer lands before the CTA's
        // shared memory is released (bounded waits), then the timeout is
        // reported
        for (int b = 0; b < a.nbuf; ++b)
          if (last_issued[b] >= 0)
            mbar_wait_bounded(smem_u32(&bars[b]), static_cast<uint32_t>(last_issued[b] / a.nbuf) & 1u);
        atomicOr(a.err, kErrWaitTimeout);
      }
      failed = true;
    }
  } else
  for (int ch = 0; ch < n_chunks; ++ch) {
    const int b = ch % a.nbuf;
    const bool ok = chunk_wait(ch, b);
    if (!__syncthreads_and(ok)) {
      if (tid == 0) {
        // let every copy still in flight land before the CTA's shared memory
        // is released, then report
        for (int cc = ch + 1; cc < n_chunks && cc < ch + a.nbuf; ++cc)
          mbar_wait_bounded(smem_u32(&bars[cc % a.nbuf]), static_cast<uint32_t>(cc / a.nbuf) & 1u);
        mbar_wait_bounded(smem_u32(&bars[b]), static_cast<uint32_t>(ch / a.nbuf) & 1u);
        atomicOr(a.err, kErrWaitTimeout);
      }
      failed = true;
      break;
    }
    const uint32_t tb = tbuf_a + static_cast<uint32_t>(b) * chunk_bytes;
    const int nt = min(a.chunk_trees, a.n_trees - ch * a.chunk_trees);
    const uint32_t la = la0 + static_cast<uint32_t>(ch & 1) * la_step;
    if constexpr (H)
      acc = nan ? walk_chunk_half<D, G, true>(tb, nt, a.tree_bytes, xa, row_bytes, acc)
                : walk_chunk_half<D, G, false>(tb, nt, a.tree_bytes, xa, row_bytes, acc);
    else if constexpr (SH > 0)
      acc = walk_chunk_split<SH, G, Q>(tbuf + (tb - tbuf_a), q, nt, a.tree_bytes, xcol, row_bytes, acc, la, a.tail,
                                       a.max_depth - SH);
    else
      acc = nan ? walk_chunk<D, G, true, Q>(tbuf + (tb - tbuf_a), q, nt, a.tree_bytes, xcol, row_bytes, acc, la)
                : walk_chunk<D, G, false, Q>(tbuf + (tb - tbuf_a), q, nt, a.tree_bytes, xcol, row_bytes, acc, la);
    if (Q > 1 && q == 0 && ch > 0) {
      // the previous chunk's leaves (complete since the last barrier)
      const uint32_t lp = la0 + static_cast<uint32_t>((ch - 1) & 1) * la_step;
      const int np = live ? a.chunk_trees : 0;  // every chunk but the last is full
      for (int t = 0; t < np; ++t) acc += lds_f32(lp + static_cast<uint32_t>(t) * row_bytes);
    }
    __syncthreads();
    if (tid == 0 && ch + a.nbuf < n_chunks) issue(ch + a.nbuf, b);
  }
  if (Q > 1 && q == 0 && !failed) {
    const uint32_t lp = la0 + static_cast<uint32_t>((n_chunks - 1) & 1) * la_step;
    const int np = live ? a.n_trees - (n_chunks - 1) * a.chunk_trees : 0;
    for (int t = 0; t < np; ++t) acc += lds_f32(lp + static_cast<uint32_t>(t) * row_bytes);
  }
  // a CTA whose wait gave up still completes its tile's bookkeeping (no
  // candidate of it valid, -inf scores): the V pass's tile count and ticket,
  // which decide when the tile offsets are scanned and the selection state
  // reset, stay consistent for this call and the next
  if (failed) acc = -INFINITY;
  pdl_trigger();
  finish_tile(a, rowidx, tile0, rows_here, count, acc, TC);
}

template <int D, int G, int Q>
__global__ void __launch_bounds__(Q <= 1 ? kFullMaxTile : 256) k_traverse_full(const __grid_constant__ TraverseArgs a) {
  traverse_full_body<D, G, Q>(a, nullptr);
}

template <int D, int G, int Q>
__global__ void __launch_bounds__(Q <= 1 ? kFullMaxTile : 256)
    k_traverse_full_dec(const __grid_constant__ TraverseArgs a, const __grid_constant__ DecodeParams d) {
  traverse_full_body<D, G, Q>(a, &d);
}

template <int D, int G, int QS>
__global__ void __launch_bounds__(256) k_traverse_half(const __grid_constant__ TraverseArgs a) {
  traverse_full_body<D, G, QS, true>(a, nullptr);
}

template <int G, int QS>
FullKernelPtr half_kernel_for(int d) {
  switch (d) {
    case 1: return k_traverse_half<1, G, QS>;
    case 2: return k_traverse_half<2, G, QS>;
    case 3: return k_traverse_half<3, G, QS>;
    case 4: return k_traverse_half<4, G, QS>;
    case 5: return k_traverse_half<5, G, QS>;
    case 6: return k_traverse_half<6, G, QS>;
    case 7: return k_traverse_half<7, G, QS>;
    case 8: return k_traverse_half<8, G, QS>;
    case 9: return k_traverse_half<9, G, QS>;
    case 10: return k_traverse_half<10, G, QS>;
    default: return nullptr;
  }
}

// Kernel of depth d (1..10) for G trees in flight and Q tree groups.
template <int G, int Q>
FullKernelPtr full_kernel_for(int d) {
  switch (d) {
    case 1: return k_traverse_full<1, G, Q>;
    case 2: return k_traverse_full<2, G, Q>;
    case 3: return k_traverse_full<3, G, Q>;
    case 4: return k_traverse_full<4, G, Q>;
    case 5: return k_traverse_full<5, G, Q>;
    case 6: return k_traverse_full<6, G, Q>;
    case 7: return k_traverse_full<7, G, Q>;
    case 8: return k_traverse_full<8, G, Q>;
    case 9: return k_traverse_full<9, G, Q>;
    case 10: return k_traverse_full<10, G, Q>;
    default: return nullptr;
  }
}

template <int G, int Q>
FullDecKernelPtr full_dec_kernel_for(int d) {
  switch (d) {
    case 1: return k_traverse_full_dec<1, G, Q>;
    case 2: return k_traverse_full_dec<2, G, Q>;
    case 3: return k_traverse_full_dec<3, G, Q>;
    case 4: return k_traverse_full_dec<4, G, Q>;
    case 5: return k_traverse_full_dec<5, G, Q>;
    case 6: return k_traverse_full_dec<6, G, Q>;
    case 7: return k_traverse_full_dec<7, G, Q>;
    case 8: return k_traverse_full_dec<8, G, Q>;
    case 9: return k_traverse_full_dec<9, G, Q>;
    case 10: return k_traverse_full_dec<10, G, Q>;
    default: return nullptr;
  }
}

// All depths and G in {2, 4, 8} for one QS (tree groups, or 0 for one group
// with the barrier-free pipeline; each QS is instantiated in its own
// translation unit, compiled in parallel).
template <int Q>
FullKernelPtr full_kernel_q(int d, int g) {
  return g == 8 ? full_kernel_for<8, Q>(d) : g == 4 ? full_kernel_for<4, Q>(d) : g == 2 ? full_kernel_for<2, Q>(d) : nullptr;
}
template <int Q>
FullDecKernelPtr full_dec_kernel_q(int d, int g) {
  return g == 8   ? full_dec_kernel_for<8, Q>(d)
         : g == 4 ? full_dec_kernel_for<4, Q>(d)
         : g == 2 ? full_dec_kernel_for<2, Q>(d)
                  : nullptr;
}

// ---------------------------------------------------------------------------
// Compact-table walk (nodes from global memory)
// ---------------------------------------------------------------------------
// Deep trees do not fit shared memory, so their nodes come from L1/L2 and
// every visit is a dependent load: the walk is latency-bound and needs many
// walks in flight per SM.  A wide feature row (1 KB at F = 256) leaves room
// for few candidates per SM, so Q lanes share one candidate: lane q of a
// candidate walks trees t0 + g*Q + q (g < G), and the G*Q leaves of each
// group are added in tree order through warp shuffles -- the same sequential
// fp32 sum as a single walker.  A warp holds 32/Q candidates.
//
// Shared memory: features [F][TC] (TC = candidates per CTA = blockDim / Q),
// then the survivor positions [TC] and the candidates' sums [TC].
__host__ __device__ inline size_t compact_smem_bytes(int F, int TC) {
  return align_up(static_cast<size_t>(F) * TC * 4, 128) + 2 * align_up(static_cast<size_t>(TC) * 4, 128);
}

template <int G, int Q>
__device__ __forceinline__ void traverse_compact_body(const TraverseArgs& a, const DecodeParams* dec) {
  extern __shared__ __align__(128) unsigned char smem[];
  constexpr int kCpw = 32 / Q;  // candidates per warp
  const int TC = blockDim.x / Q;
  const int tid = threadIdx.x;
  const long long tile0 = static_cast<long long>(blockIdx.x) * TC;
  pdl_wait();
  if (a.stream && *reinterpret_cast<volatile const unsigned*>(&a.stream->done)) return;
  const long long count = a.p_pass ? static_cast<long long>(a.state->survivors) : a.n;
  if (tile0 >= count) return;
  const int rows_here = static_cast<int>(min(static_cast<long long>(TC), count - tile0));

  float* xs = reinterpret_cast<float*>(smem);
  const size_t rows_off = align_up(static_cast<size_t>(a.F) * TC * 4, 128);
  uint32_t* rowidx = reinterpret_cast<uint32_t*>(smem + rows_off);
  float* sums = reinterpret_cast<float*>(smem + rows_off + align_up(static_cast<size_t>(TC) * 4, 128));
  if (a.p_pass && tid < rows_here) rowidx[tid] = a.rows[tile0 + tid];
  // threads [0, TC) stage one row each; feature rows are read once, the node
  // tables are re-read by every tile
  __syncthreads_or(tid < TC && stage_row(a, dec, xs, rowidx, tile0, rows_here, TC, true));

  const int lane = tid & 31, warp = tid >> 5;
  const int cl = lane % kCpw;       // candidate within the warp
  const int q = lane / kCpw;        // this lane's share of each tree group
  const int c = warp * kCpw + cl;   // candidate within the tile
  float acc = 0.0f;
  if (warp * kCpw < rows_here) {    // warp-uniform: a warp past the rows idles
    const uint32_t* offs = reinterpret_cast<const uint32_t*>(a.table);
    const uint2* recs =
        reinterpret_cast<const uint2*>(a.table + align_up(static_cast<size_t>(a.n_trees) * 4, 16));
    const unsigned long long keep = policy_evict_last();
    const float* xc = xs + c;
    const int steps = a.max_depth + 1;
    for (int t0 = 0; t0 < a.n_trees; t0 += G * Q) {
      const uint2* tr[G];
      uint32_t j[G];
      bool live[G];
      uint2 r[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const int t = t0 + g * Q + q;
        live[g] = t < a.n_trees;
        tr[g] = recs + (live[g] ? __ldg(offs + t) : 0u);
        j[g] = 0;
      }
      for (int s = 0; s < steps; ++s) {
        // all G node loads, then the decisions; a walk at its leaf stays
        // there (its record is re-read, a leaf's feature field is 0)
#pragma unroll
        for (int g = 0; g < G; ++g) r[g] = ldg_u2_hint(tr[g] + j[g], keep);
        bool any = false;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const uint32_t meta = r[g].y;
          const float x = xc[(meta & kCompactFeatureMask) * TC];
          uint32_t right = x >= __uint_as_float(r[g].x) ? 1u : 0u;
          if ((x != x) && !(meta & kMetaDefaultLeft)) right = 1u;
          const bool move = live[g] && !(meta & kMetaLeaf);
          j[g] = move ? ((meta >> kCompactChildShift) & kCompactChildMask) + right : j[g];
          any |= move;
        }
        if (!__any_sync(0xFFFFFFFFu, any)) break;  // every walk of the warp is at a leaf
      }
      // r[g] is each walk's leaf record.  Tree t0 + g*Q + qq of candidate c
      // sits in lane qq*kCpw + cl: add them in tree order.
#pragma unroll
      for (int g = 0; g < G; ++g) {
#pragma unroll
        for (int qq = 0; qq < Q; ++qq) {
          const float v = __shfl_sync(0xFFFFFFFFu, __uint_as_float(r[g].x), qq * kCpw + cl);
          if (t0 + g * Q + qq < a.n_trees) acc += v;
        }
      }
    }
  }
  if (q == 0) sums[c] = acc;
  __syncthreads();
  pdl_trigger();
  finish_tile(a, rowidx, tile0, rows_here, count, tid < TC ? sums[tid] : 0.0f, TC);
}

template <int G, int Q>
__global__ void __launch_bounds__(256) k_traverse_compact(const __grid_constant__ TraverseArgs a) {
  traverse_compact_body<G, Q>(a, nullptr);
}

template <int G, int Q>
__global__ void __launch_bounds__(256)
    k_traverse_compact_dec(const __grid_constant__ TraverseArgs a, const __grid_constant__ DecodeParams d) {
  traverse_compact_body<G, Q>(a, &d);
}

}  // namespace walk
}  // namespace mlt
