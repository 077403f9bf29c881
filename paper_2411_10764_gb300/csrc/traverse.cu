// Launch planning and the plain (stored-feature) tree-walk kernels.  The
// device code lives in walk.cuh; traverse_dec.cu instantiates the variants
// that build features from candidate indices.
#include <algorithm>
#include <cmath>

#include "walk.cuh"

namespace mlt {
namespace {

using namespace walk;

constexpr size_t kSmPerSm = 228 * 1024;  // shared memory per SM
constexpr size_t kCtaReserve = 1024;     // reserved per resident CTA
constexpr size_t kStaticSmem = 512;      // finish_tile and scan_tiles statics

}  // namespace

FullKernelPtr full_kernel_q1(int depth, int group) { return full_kernel_q<1>(depth, group); }

FullKernelPtr full_kernel(int depth, int group, int q) {
  switch (q) {
    case 0: return full_kernel_sf(depth, group);
    case 1: return full_kernel_q1(depth, group);
    case 2: return full_kernel_q2(depth, group);
    case 4: return full_kernel_q4(depth, group);
    default: return nullptr;
  }
}

// Choose candidates per CTA (threads), trees per shared-memory chunk, chunk
// buffers and trees walked together (group) for a full table.  Rules (from
// sweeps of every shape on the five workloads):
//   * every CTA re-streams the whole table through shared memory, and with
//     small CTAs the stream (not the walk) sets the pace, so CTAs hold 256
//     candidates unless the batch would then occupy fewer than a quarter of
//     the SMs; then the largest size that reaches that is used;
//   * when the busiest SM holds two or more tiles, a shape that keeps two
//     CTAs resident (twice the warps to hide shared-memory latency) beats
//     one CTA with bigger chunks: take the largest chunk that still allows
//     two; otherwise one CTA with the largest chunk (fewest barriers);
//   * a thread walks 8 trees at once (4 with tree groups when more than 8
//     warps share the SM), the chunk permitting;
//   * a batch of under 32 (64) candidates per SM splits each tile's trees
//     over 4 (2) groups of warps;
//   * one CTA per SM whose chunks hold fewer than 8 trees grows past 256
//     candidates, up to 384 (below).
ScreenShape plan_full(int F, int n_trees, uint32_t tb, long long n_eff, int sms, int optin,
                      const ShapeOverride& ov, bool half) {
  if (sms < 1) sms = 1;
  if (n_eff < 1) n_eff = 1;
  // tree groups per CTA: a batch of less than a warp (or two) per SM gets
  // its trees split over 4 (2) groups of warps; half tables walk with one
  const int q = half ? 1 : ov.lanes ? ov.lanes : n_eff < 32LL * sms ? 4 : n_eff < 64LL * sms ? 2 : 1;
  if (q != 1 && q != 2 && q != 4) return ScreenShape{};
  if (half && ov.lanes > 1) return ScreenShape{};
  const int xb = half ? 2 : 4;  // bytes per staged feature
  auto smem_of = [&](int tc, int chunk, int nb) {
    return full_smem_bytes(F, tc, nb, static_cast<uint32_t>(chunk) * tb, q, chunk, xb);
  };
  auto fits = [&](size_t smem) { return smem + kStaticSmem <= static_cast<size_t>(optin); };
  auto resident = [&](size_t smem, int tc) {
    return static_cast<int>(std::min<size_t>(
        {kSmPerSm / (smem + kStaticSmem + kCtaReserve), static_cast<size_t>(2048 / (tc * q)), 32}));
  };
  int tc = 256 / q;
  if (!ov.threads) {
    while (tc > 32 && (n_eff + tc - 1) / tc < (sms + 3) / 4) tc >>= 1;
    // wide rows: shrink the tile until it fits with the smallest chunk
    while (tc > 32 && !fits(smem_of(tc, 1, 2))) tc >>= 1;
    // spread the tiles evenly: the smallest multiple of 32 (at least 64)
    // that gives the busiest SM no more tiles; decided before the chunk
    // size, which the smaller tile may let grow
    const long long t_sm = ((n_eff + tc - 1) / tc + sms - 1) / sms;
    const long long per_tile = (n_eff + sms * t_sm - 1) / (sms * t_sm);
    const int tb = static_cast<int>(std::min<long long>(tc, (per_tile + 31) / 32 * 32));
    if (tb >= 64) tc = tb;
  } else {
    tc = ov.threads;
  }
  if (tc * q > (q == 1 && !half ? kFullMaxTile : 256)) return ScreenShape{};
  const long long tiles = (n_eff + tc - 1) / tc;
  const long long tiles_sm = (tiles + sms - 1) / sms;
  ScreenShape best{};
  int best_rank = -1;
  for (int ch : {16, 8, 4, 2, 1}) {
    if (ov.chunk_trees && ch != ov.chunk_trees) continue;
    const int chunk = std::min(ch, n_trees);
    for (int nb : {2, 3}) {
      if (ov.nbuf && nb != ov.nbuf) continue;
      const size_t smem = smem_of(tc, chunk, nb);
      if (!fits(smem)) continue;
      const int res = std::min<long long>(resident(smem, tc), tiles_sm);
      // rank: two resident CTAs when there are two tiles to run, then
      // chunk size, then fewer buffers
      const int want2 = tiles_sm >= 2 && res >= 2 ? 1 : 0;
      const int rank = want2 * 1000 + chunk * 10 + (3 - nb);
      if (rank > best_rank) {
        best_rank = rank;
        const int warps = res * tc * q / 32;
        int group = q == 1 || warps <= 8 ? 8 : 4;
        if (ov.group) group = ov.group;
        // each group walks chunk / q trees of a chunk
        const int per = std::max(1, chunk / q);
        group = std::min(group, per >= 8 ? 8 : per >= 4 ? 4 : 2);
        best.threads = tc;
        best.lanes = q;
        best.chunk_trees = chunk;
        best.nbuf = nb;
        best.group = group;
        best.smem = smem;
        best.p_grid = sms * std::max(1, res);  // CTAs per wave: the tiles an SM gets, up to residency
        best.resident = std::max(1, res);
        best.sync_free = q == 1 && best.resident == 1 ? 1 : 0;
      }
    }
  }
  // one CTA of 256 candidates per SM, no tree groups, fewer than 8 trees in
  // flight per thread (large trees: the chunk holds few): the walk waits on
  // its dependent shared-memory reads, so grow the tile (more warps) while
  // the same chunks still fit and the busiest SM keeps two or more tiles.
  // Measured on workload 4 (depth 10, 4-tree chunks, 96 decoded features):
  // V pass 9.67 / 9.48 / 8.66 / 7.93 / 7.36 ms at 256 / 288 / 320 / 352 /
  // 384 candidates.  With 8 trees in flight the shared-memory pipe is
  // already busy, and a larger tile was slower (workload 3: 2.00 ms at 256
  // candidates, 2.19 ms at 288).
  if (best.threads == 256 && q == 1 && !half && best.resident == 1 && best.group < 8 && !ov.threads) {
    for (int t2 = kFullMaxTile; t2 > 256; t2 -= 32) {
      const size_t smem = smem_of(t2, best.chunk_trees, best.nbuf);
      if (!fits(smem) || (n_eff + t2 - 1) / t2 < 2LL * sms) continue;
      best.threads = t2;
      best.smem = smem;
      break;
    }
  }
  return best;  // threads == 0: nothing fits
}

// Split table (deep trees): the same tile and chunk pipeline as a full
// table, streaming head blocks of hb bytes.  A warp's walk over a group of
// trees lasts as long as its deepest path, which waits on one L2 round trip
// per level below the head, so the shape maximises latency hiding per
// candidate of the busiest SM.  Measured on GB300 (F = 256, 1,000-2,000
// trees of depth <= 12): warps per SM count more than trees in flight per
// thread (16 warps x 4 trees beat 8 warps x 8 trees by 1.24x), and a tree
// group whose share of a chunk holds fewer than G trees wastes the rest
// (8-tree chunks over 4 groups ran 1.7x slower than 16-tree chunks), and
// two resident CTAs beat one CTA with the same warps (their chunk pipelines
// do not meet at each other's barriers: 64 candidates x 8 groups x 2 CTAs
// ran 8 % faster than 128 x 8 x 1).  The rule minimises
//   tiles of the busiest SM x candidates per tile
//     / (warps per SM x trees in flight per thread ^ 0.7)
//     x (1 + 8 / tile) x (0.85 with two or more resident CTAs),
// the tile factor for the head blocks every tile re-streams.  Up to 512
// threads per CTA (1,024 with 8 tree groups: the split kernels' launch
// bounds); registers (56-88 a thread) bound the warps an SM holds.
ScreenShape plan_split(int F, int n_trees, uint32_t hb, long long n_eff, int sms, int optin,
                       const ShapeOverride& ov) {
  if (sms < 1) sms = 1;
  if (n_eff < 1) n_eff = 1;
  ScreenShape best{};
  double best_cost = 1e300;
  for (int q : {1, 2, 4, 8}) {
    if (ov.lanes && q != ov.lanes) continue;
    for (int tc : {256, 128, 64, 32}) {
      if (ov.threads && tc != ov.threads) continue;
      if (tc * q > (q == 8 ? 1024 : 512)) continue;
      for (int ch : {32, 16, 8, 4}) {
        if (ov.chunk_trees && ch != ov.chunk_trees) continue;
        const int chunk = std::min(ch, n_trees);
        for (int nb : {2, 3}) {
          if (ov.nbuf && nb != ov.nbuf) continue;
          const size_t smem = full_smem_bytes(F, tc, nb, static_cast<uint32_t>(chunk) * hb, q, chunk);
          if (smem + kStaticSmem > static_cast<size_t>(optin)) continue;
          for (int g : {8, 4, 2}) {
            if (ov.group && g != ov.group) continue;
            if (!ov.group && g > std::max(2, chunk / q)) continue;  // idle tree slots
            const int regs = g == 8 ? 88 : g == 4 ? 64 : 56;
            const long long tiles = (n_eff + tc - 1) / tc;
            const long long tiles_sm = (tiles + sms - 1) / sms;
            const int fit = static_cast<int>(std::min<size_t>(
                {kSmPerSm / (smem + kStaticSmem + kCtaReserve), static_cast<size_t>(2048 / (tc * q)),
                 static_cast<size_t>(65536 / (tc * q * regs)), 32}));
            if (fit < 1) continue;
            const int res = static_cast<int>(std::min<long long>(fit, tiles_sm));
            // tree groups with no tree of a chunk idle
            const double warps = static_cast<double>(res) * tc * std::min(q, chunk) / 32.0;
            const double gg = std::min(g, std::max(1, chunk / q));
            const double cost = static_cast<double>(tiles_sm) * tc / (warps * std::pow(gg, 0.7)) * (1.0 + 8.0 / tc) *
                                (res >= 2 ? 0.85 : 1.0) * (g > gg ? 1.05 : 1.0);
            if (cost < best_cost * (1.0 - 1e-9)) {
              best_cost = cost;
              best.threads = tc;
              best.lanes = q;
              best.chunk_trees = chunk;
              best.nbuf = nb;
              best.group = g;
              best.smem = smem;
              best.p_grid = sms * std::max(1, res);
              best.resident = std::max(1, res);
              best.sync_free = q == 1 && best.resident == 1 ? 1 : 0;
            }
          }
        }
      }
    }
  }
  return best;
}

ScreenShape cap_residency(const ScreenShape& s, int optin) {
  if (s.threads == 0 || s.resident < 1) return s;
  const size_t per_cta = kStaticSmem + kCtaReserve;
  const size_t fit = kSmPerSm / (s.smem + per_cta);
  if (fit <= static_cast<size_t>(s.resident)) return s;
  // resident + 1 CTAs of this size cannot fit, whatever the per-CTA
  // overheads are
  const size_t need = kSmPerSm / (s.resident + 1) + 1;
  ScreenShape c = s;
  if (need + kStaticSmem <= static_cast<size_t>(optin)) c.smem = std::max(s.smem, (need + 15) & ~static_cast<size_t>(15));
  return c;
}

// Deep-tree walk: candidates per CTA (TC), lanes per candidate (Q) and trees
// in flight per lane (G).  Every visit waits on an L1/L2 load, so a
// candidate's walk takes time in proportion to its trees / (Q * G), and an SM
// finishes (resident CTAs * TC * Q * G) walks in flight at a time.  Measured
// on GB300 (F = 256, 1,000-2,000 trees of depth <= 12): throughput grows
// with the walks in flight up to about 3,072 per SM and falls beyond it, as
// the trees in flight crowd L1.  So the rule minimises
//   (candidates per SM) / (walks in flight, counted up to 3,072 and
//                          discounted by a quarter of any excess)
// where resident CTAs are limited by shared memory (F * TC * 4 bytes of
// features), 2,048 threads, registers (48 a thread at G = 4, 64 at G = 8)
// and the tiles the batch gives each SM.  Ties go to fewer lanes (fewer
// bank conflicts on the feature gathers), then to larger CTAs.
ScreenShape plan_compact(int F, long long n_eff, int sms, int optin, const ShapeOverride& ov) {
  constexpr double kSaturation = 3072.0;
  ScreenShape best{};
  double best_cost = 1e300;
  if (sms < 1) sms = 1;
  if (n_eff < 1) n_eff = 1;
  for (int q : {1, 2, 4, 8}) {
    if (ov.lanes && q != ov.lanes) continue;
    for (int tc : {256, 128, 64, 32, ov.threads}) {
      if (tc == 0 || (ov.threads && tc != ov.threads)) continue;
      const int threads = tc * q;
      if (threads > 256) continue;
      const size_t smem = compact_smem_bytes(F, tc);
      if (smem + kStaticSmem > static_cast<size_t>(optin)) continue;
      for (int g : {8, 4}) {
        if (ov.group && g != ov.group) continue;
        const int regs = g == 8 ? 64 : 48;
        const int ctas_sm = static_cast<int>(std::min<size_t>(
            {kSmPerSm / (smem + kStaticSmem + kCtaReserve), static_cast<size_t>(2048 / threads),
             static_cast<size_t>(65536 / (threads * regs)), 32}));
        if (ctas_sm < 1) continue;
        const long long tiles = (n_eff + tc - 1) / tc;
        const long long tiles_sm = (tiles + sms - 1) / sms;
        const int resident = static_cast<int>(std::min<long long>(ctas_sm, tiles_sm));
        const double inflight = static_cast<double>(resident) * threads * g;
        const double eff = inflight <= kSaturation ? inflight
                                                   : std::max(kSaturation - 0.25 * (inflight - kSaturation), 256.0);
        const double cost = static_cast<double>(tiles_sm) * tc / eff;
        if (cost < best_cost * (1.0 - 1e-9)) {
          best_cost = cost;
          best.threads = tc;
          best.lanes = q;
          best.group = g;
          best.smem = smem;
        }
      }
    }
  }
  return best;
}

namespace {
using CompactKernel = void (*)(TraverseArgs);
CompactKernel compact_kernel(int group, int lanes) {
  if (group == 8) {
    switch (lanes) {
      case 1: return k_traverse_compact<8, 1>;
      case 2: return k_traverse_compact<8, 2>;
      case 4: return k_traverse_compact<8, 4>;
      case 8: return k_traverse_compact<8, 8>;
    }
  } else if (group == 4) {
    switch (lanes) {
      case 1: return k_traverse_compact<4, 1>;
      case 2: return k_traverse_compact<4, 2>;
      case 4: return k_traverse_compact<4, 4>;
      case 8: return k_traverse_compact<4, 8>;
    }
  }
  return nullptr;
}
}  // namespace

cudaError_t launch_traverse(const DeviceModel& m, const TraverseArgs& args, const ScreenShape& shape,
                            long long n_tiles, cudaStream_t st) {
  if (n_tiles <= 0) return cudaSuccess;
  // full-table P pass: whole waves of CTAs, the survivors split evenly over
  // them on the device (CTAs without rows exit at once)
  TraverseArgs a = args;
  long long ctas = n_tiles;
  if (args.p_pass && m.kind != kTableCompact && shape.p_grid > 0) {
    a.p_wave = shape.p_grid;
    ctas = (n_tiles + shape.p_grid - 1) / shape.p_grid * shape.p_grid;
  }
  const dim3 grid(static_cast<unsigned>(ctas));
  if (m.kind != kTableCompact) {
    const int q = shape.sync_free ? 0 : shape.lanes;
    FullKernelPtr k = m.kind == kTableHalf
                          ? (shape.lanes == 1 ? half_kernel(m.depth, shape.group, shape.sync_free != 0) : nullptr)
                      : m.kind == kTableSplit ? split_kernel(m.head_levels, shape.group, q)
                                              : full_kernel(m.depth, shape.group, q);
    if (k == nullptr) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(shape.smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(k, grid, dim3(shape.threads * shape.lanes), shape.smem, st, a);
    if (e != cudaSuccess) return e;
  } else {
    CompactKernel k = compact_kernel(shape.group, shape.lanes);
    if (k == nullptr) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(shape.smem));
    if (e != cudaSuccess) return e;
    e = launch_pdl(k, grid, dim3(shape.threads * shape.lanes), shape.smem, st, a);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace mlt
