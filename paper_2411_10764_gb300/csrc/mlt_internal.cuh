// Internal declarations shared by the libmlt translation units (not part of
// the C ABI).  Device table formats, launch descriptors and launchers.
#pragma once

#include <cstddef>
#include <cstdint>
#include <utility>
#include <cuda_runtime.h>

namespace mlt {

constexpr int kMaxKnobs = 16;
constexpr int kMaxOptions = 256;
constexpr int kMaxProgram = 256;
constexpr int kMaxF = 1024;
constexpr int kMaxK = 16384;
constexpr int kMaxDepth = 14;  // model A of the paper has depth 14 (Table 3)
constexpr int kFullMaxTile = 384;  // candidates of a full-table tile walked by one group of warps
constexpr int kMaxFullDepth = 10;  // deeper ensembles use the compact table

// Device error bits (accumulated in one word, read by mlt_sync_status).
constexpr unsigned kErrWaitTimeout = 1u;  // an mbarrier wait gave up
constexpr unsigned kErrSelect = 2u;       // top-k bookkeeping out of range
constexpr unsigned kErrBadIndex = 4u;     // a rerank candidate index outside [0, n)

// A bounded device wait gives up after this many nanoseconds.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// ---------------------------------------------------------------------------
// Packed device tables
// ---------------------------------------------------------------------------
// Full table (depth D <= kMaxFullDepth): every tree is stored as a complete
// binary tree of depth D, `tree_bytes` apart (a multiple of 16).  A node has
// a threshold (float), a feature index (< kMaxF) and a NaN-goes-left flag;
// its heap index is j (children 2j+1, 2j+2).  Each level is laid out for the
// way a warp reads it (FullLayout below):
//   levels [0, top)  : 8-byte records {threshold, meta} with meta = feature
//                      | flag << 31 -- few distinct nodes, mostly broadcast
//                      reads;
//   levels [top, D)  : the thresholds as a 4-byte array and the metas as a
//                      2-byte array (feature | flag << 15) -- 32-lane
//                      gathers; 6 bytes a node where 8-byte records would
//                      take 8, so more candidates and trees fit in shared
//                      memory at once;
//   then the 2^D leaves (4 bytes each, leaf i = child heap index - (2^D - 1)).
// A shallower leaf is replicated into every leaf slot below it (its
// pass-through nodes test feature 0; any path gives the leaf).
//
// Compact table (any depth <= kMaxDepth): uint32 offsets[n_trees] (in
// records, from the start of the record area, which begins at byte
// align16(4 * n_trees)), then each tree's existing nodes in breadth-first
// order as {float value; uint32 meta}:
//   meta bit 30 = leaf (value = leaf output), bit 31 = NaN goes left,
//   bits 10..29 = index of the left child within the tree (right = left+1),
//   bits 0..9 = feature index (F <= 1024).
//
// Half table (depth D <= kMaxFullDepth, loaded by mlt_load_ensemble_f16):
// the full table's heap with thresholds and leaves rounded to IEEE binary16
// (round to nearest even), `tree_bytes` apart:
//   levels [0, D-1)  : 4-byte words {bits 0..15 threshold (binary16), bits
//                      16..25 feature index, bit 31 NaN goes left};
//   level D-1 (last) : 8-byte records {that word; left leaf | right leaf << 16
//                      (binary16)}.
// The features are rounded to binary16 when staged, so a candidate is
// compared and scored exactly as the rounded model scores the rounded row.
//
// Split table (models V and P deeper than kMaxFullDepth): each tree's first
// H levels as a complete heap that streams through shared memory like a
// full table, and the rest as compact records read from global memory:
//   every node sends a missing value right: a node whose missing values go
//   left has its subtrees swapped, threshold -prev(t) and bit 31 of its meta
//   set ("negate": the walk compares -x), so x < t (or missing) becomes
//   -x >= -prev(t) (or missing), an unordered >= with no missing-value test;
//   head block (split_head_bytes(H) bytes, one per tree, contiguous):
//     heap slots 0 .. 2^H - 2 (levels 0 .. H-1): 8-byte {threshold, meta}
//       with meta = feature | negate bit (bit 31); a slot on or below a
//       shallower leaf is a pass-through {0, 0} (every exit below it holds
//       that leaf, so the direction taken does not matter);
//     heap slots 2^H - 1 .. 2^(H+1) - 2 (level H, the exits): a leaf
//       {value, kMetaLeaf} or the level-H split node itself in the compact
//       format, its child index counted from the tree's tail base;
//     last 8 bytes: {tail base (record index into the tail array), 0};
//   tail array (after the n_trees head blocks, 16-byte aligned): every
//     tree's nodes below level H in breadth-first order, compact records
//     (children adjacent, right = left + 1).
// The walk reads H levels and the exit from shared memory; only paths that
// go deeper than H touch global memory (L2-resident: evict_last).
enum TableKind : int { kTableFull = 0, kTableCompact = 1, kTableHalf = 2, kTableSplit = 3 };

constexpr int kSplitHeadDefault = 6;  // head levels of a split table (6 or 7)
__host__ __device__ constexpr uint32_t split_head_bytes(int H) { return (2u << H) * 8u; }

struct HalfLayout {
  uint32_t n_inner;   // nodes in levels [0, D-1)
  uint32_t off_last;  // byte offset of the last-level 8-byte records
  uint32_t bytes;     // bytes per tree (multiple of 16)
};

__host__ __device__ constexpr HalfLayout half_layout(int D) {
  const uint32_t n_inner = (1u << (D - 1)) - 1u;
  const uint32_t off_last = (n_inner * 4u + 7u) & ~7u;
  const uint32_t bytes = (off_last + (1u << (D - 1)) * 8u + 15u) & ~15u;
  return HalfLayout{n_inner, off_last, bytes};
}

constexpr uint32_t kHalfFeatureShift = 16;
constexpr uint32_t kHalfFeatureMask = 0x3FFu;

struct FullLayout {
  uint32_t top;       // levels held as 8-byte records
  uint32_t n_top;     // nodes in levels [0, top)
  uint32_t n_inner;   // nodes in levels [0, D)
  uint32_t off_thr;   // byte offset of the thresholds of levels [top, D)
  uint32_t off_meta;  // byte offset of their 2-byte metas
  uint32_t off_leaf;  // byte offset of the 2^D leaves
  uint32_t bytes;     // bytes per tree (multiple of 16)
};

__host__ __device__ constexpr FullLayout full_layout(int D) {
  const uint32_t top = D - 1 < 4 ? static_cast<uint32_t>(D - 1) : 4u;
  const uint32_t n_top = (1u << top) - 1u;
  const uint32_t n_inner = (1u << D) - 1u;
  const uint32_t off_thr = n_top * 8u;
  const uint32_t off_meta = off_thr + (n_inner - n_top) * 4u;
  const uint32_t off_leaf = (off_meta + (n_inner - n_top) * 2u + 3u) & ~3u;
  const uint32_t bytes = (off_leaf + (1u << D) * 4u + 15u) & ~15u;
  return FullLayout{top, n_top, n_inner, off_thr, off_meta, off_leaf, bytes};
}
constexpr uint32_t kMeta16Feature = 0x7FFFu;  // 2-byte meta: feature index
constexpr uint32_t kMeta16Left = 0x8000u;     // 2-byte meta: NaN goes left
static_assert(kMaxF <= static_cast<int>(kMeta16Feature) + 1, "feature index must fit a 2-byte meta");

constexpr uint32_t kMetaLeaf = 1u << 30;
constexpr uint32_t kMetaDefaultLeft = 1u << 31;
constexpr uint32_t kCompactFeatureMask = 0x3FFu;  // bits 0..9
constexpr uint32_t kCompactChildShift = 10;       // bits 10..29
constexpr uint32_t kCompactChildMask = 0xFFFFFu;

struct DeviceModel {
  const unsigned char* table = nullptr;
  size_t bytes = 0;
  int kind = kTableFull;
  int n_trees = 0;
  int depth = 0;
  uint32_t tree_bytes = 0;  // full and half tables: bytes per tree; split tables: head block bytes
  int head_levels = 0;      // split tables: H
  const unsigned char* tail = nullptr;  // split tables: the tail records
  size_t tail_off = 0;                  // split tables: byte offset of the tail records
};

// ---------------------------------------------------------------------------
// Knob decoder (kernel parameter; ~5.3 KB)
// ---------------------------------------------------------------------------
struct DecodeParams {
  int n_knobs;
  int F;
  long long first_index;
  const long long* index_list;  // device: candidate of position i (null: first_index + i)
  int radix[kMaxKnobs];
  int opt_off[kMaxKnobs];
  float opts[kMaxOptions];
  int op[kMaxProgram];
  int a[kMaxProgram];
  int b[kMaxProgram];
  float c[kMaxProgram];
};

// ---------------------------------------------------------------------------
// Scratch and top-k selection state
// ---------------------------------------------------------------------------
// The P pass histograms the top kTopBits bits of every rank key; the top-k
// kernel reads it to find the bucket holding the k-th key, collects the keys
// of that bucket and above (a few hundred to a few thousand here), and one
// CTA narrows them to exactly k by radix digits and orders those.
constexpr int kTopBits = 12;
constexpr int kTopBins = 1 << kTopBits;

struct SelectState {
  unsigned int survivors;  // valid candidates of the current batch
  unsigned int n_cand;     // keys collected for the final sort
  unsigned int ticket;     // CTAs of the top-k kernel that finished
  unsigned int v_ticket;   // CTAs of the V pass that finished
  unsigned int hist[kTopBins];  // 16-byte aligned
};

// Batched accumulation (mlt_screen_until): bookkeeping carried on the device
// across the batches of one call.  Once `done` is set, every later batch's
// kernels return at once (no host round trip decides when to stop).
struct StreamState {
  unsigned int total;           // survivors accumulated so far
  unsigned int done;            // the target count was reached
  unsigned int batches;         // batches screened
  unsigned int pad;
  unsigned long long consumed;  // candidates screened
};

struct Scratch {
  uint32_t* masks = nullptr;         // [ceil(n/32)] validity ballots
  uint32_t* tile_counts = nullptr;   // [n_tiles] survivors per V tile
  uint32_t* tile_offsets = nullptr;  // [n_tiles] exclusive prefix
  uint32_t* rows = nullptr;          // [n] survivor positions, ascending
  unsigned long long* keys = nullptr;  // [n] (score, position) keys
  unsigned long long* cand = nullptr;  // [n] collected keys
  SelectState* state = nullptr;
  unsigned int* err = nullptr;       // device error word
};

// ---------------------------------------------------------------------------
// Launch descriptors
// ---------------------------------------------------------------------------
struct TraverseArgs {
  uint32_t* tile_offsets;  // V pass: exclusive prefix of tile_counts (last CTA)
  SelectState* state_rw;   // V pass: written by the last CTA
  // candidates
  const float* feats;      // [n][F] (null when decoding)
  int F;
  long long n;             // candidates of the batch (V pass)
  int p_pass;              // 0: V pass over all rows; 1: P pass over survivors
  int vec4;                // feature rows 16-byte aligned and F % 4 == 0
  const uint32_t* rows;    // P pass: survivor positions
  const SelectState* state;  // P pass: survivor count
  // trees
  const unsigned char* table;
  int n_trees;
  uint32_t tree_bytes;     // full table
  int chunk_trees;         // full table: trees per shared-memory chunk
  int nbuf;                // full table: chunk buffers
  int max_depth;           // compact and split tables
  const uint2* tail;       // split tables: the tail records
  float tau;
  // outputs
  float* out_pvalid;
  float* out_perf;
  uint32_t* masks;
  uint32_t* tile_counts;
  unsigned long long* keys;
  unsigned int* hist;      // P pass: key histogram (kTopBins)
  unsigned int* err;
  int decode;              // features built from candidate indices
  // batched accumulation (null: a single batch)
  StreamState* stream;
  long long pos_base;      // position of the batch's first candidate in the call
  int p_wave;              // full-table P pass: CTAs one wave holds (0: the grid)
  // failure-detection self-test (full tables): CTA `stall_cta` waits for its
  // first chunk on a barrier phase that nothing completes and gives up after
  // stall_ns (-1: no CTA does)
  int stall_cta = -1;
  unsigned long long stall_ns = 0;
};

struct ScreenShape {
  int threads;         // candidates per CTA
  size_t smem;         // dynamic shared memory bytes
  int chunk_trees;
  int nbuf;
  int group;           // trees walked together per thread (ILP)
  int lanes = 1;       // threads sharing one candidate's trees: warp groups (full tables) or
                       // lanes of a warp (compact tables); CTA = threads * lanes
  int p_grid = 0;      // full-table P pass: CTAs one wave holds (resident per SM x SMs)
  int sync_free = 0;   // full tables, one tree group: barrier-free chunk pipeline (one CTA per SM)
  int resident = 0;    // full tables: CTAs meant to share an SM (shared memory is padded so
                       // that no more fit: the block scheduler would otherwise stack tiles
                       // on some SMs and leave others idle)
};

// Launch-shape override (mlt_tune_walk): 0 fields mean "choose".
struct ShapeOverride {
  int threads = 0;      // candidates per CTA
  int chunk_trees = 0;
  int nbuf = 0;
  int lanes = 0;        // splits
  int group = 0;
};

// Full-table walk kernels for Q tree groups (Q = 1, 2 or 4), G in {2, 4, 8}
// trees in flight, depth 1..10: traverse.cu / traverse_dec.cu (Q = 1),
// traverse_q2.cu (Q = 2), traverse_q4.cu (Q = 4).  nullptr if not built.
using FullKernelPtr = void (*)(TraverseArgs);
using FullDecKernelPtr = void (*)(TraverseArgs, DecodeParams);
// q = tree groups (1, 2, 4), or 0 for one group with the barrier-free
// chunk pipeline
FullKernelPtr full_kernel(int depth, int group, int q);
FullDecKernelPtr full_dec_kernel(int depth, int group, int q);
FullKernelPtr full_kernel_q1(int depth, int group);
FullDecKernelPtr full_dec_kernel_q1(int depth, int group);
FullKernelPtr full_kernel_q2(int depth, int group);
FullDecKernelPtr full_dec_kernel_q2(int depth, int group);
FullKernelPtr full_kernel_q4(int depth, int group);
FullDecKernelPtr full_dec_kernel_q4(int depth, int group);
// traverse_sf.cu: one tree group, barrier-free chunk pipeline
FullKernelPtr full_kernel_sf(int depth, int group);
FullDecKernelPtr full_dec_kernel_sf(int depth, int group);
// traverse_half.cu: half tables (one tree group, stored features only)
FullKernelPtr half_kernel(int depth, int group, bool sync_free);
// traverse_split.cu: split tables, H head levels, q tree groups (0: one
// group, barrier-free pipeline), G in {4, 8}
FullKernelPtr split_kernel(int head_levels, int group, int q);
FullDecKernelPtr split_dec_kernel(int head_levels, int group, int q);

// traverse.cu
// n_eff: candidates the pass is expected to walk (used for load balance).
// half: a half table (binary16 features staged, one tree group)
ScreenShape plan_full(int F, int n_trees, uint32_t tree_bytes, long long n_eff, int sms,
                      int device_smem_optin, const ShapeOverride& ov, bool half);
ScreenShape plan_compact(int F, long long n_eff, int sms, int device_smem_optin,
                         const ShapeOverride& ov);
// split tables: head blocks of hb bytes
ScreenShape plan_split(int F, int n_trees, uint32_t hb, long long n_eff, int sms, int device_smem_optin,
                       const ShapeOverride& ov);
// Pad a full-table shape's shared memory so that at most s.resident CTAs fit
// on an SM.
ScreenShape cap_residency(const ScreenShape& s, int optin);
cudaError_t launch_traverse(const DeviceModel& m, const TraverseArgs& args,
                            const ScreenShape& shape, long long n_tiles, cudaStream_t st);
// traverse_dec.cu
cudaError_t launch_traverse_dec(const DeviceModel& m, const TraverseArgs& args,
                                const DecodeParams& dec, const ScreenShape& shape,
                                long long n_tiles, cudaStream_t st);
cudaError_t launch_decode_rows(const DecodeParams& dec, long long n, uint8_t* out_knobs,
                               float* out_feats, cudaStream_t st);
// Decoded batches of at least this many candidates build their rows with the
// compiled feature program by default (mlt_tune_decode_jit changes it).
constexpr long long kDecodeJitMinN = 1LL << 20;
// jit_decode.cu: the feature program compiled at run time (NVRTC) into a
// decode kernel that writes rows [n][F]; fn is null when that is
// unavailable (why says why)
struct JitDecoder {
  void* fn;
  int tc;
  size_t smem;
  const char* why;
};
JitDecoder jit_decoder_for(const DecodeParams& d, int dev);
bool jit_available();
cudaError_t launch_jit_decode(const JitDecoder& jd, const DecodeParams& d, long long n, float* out,
                              cudaStream_t st);

// Launch with programmatic dependent launch allowed: the kernel may start
// while the previous kernel on the stream finishes; it must execute
// pdl_wait() before it touches anything that kernel (or any earlier one)
// writes, and pdl_trigger() once its own dependents may be scheduled.
template <typename... K, typename... A>
cudaError_t launch_pdl(void (*kernel)(K...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       A&&... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<A>(args)...);
}

#ifdef __CUDACC__
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
#endif

// select.cu
cudaError_t launch_compact(const Scratch& s, long long n, int tile, long long n_tiles,
                           const StreamState* ss, cudaStream_t st);
// count: survivors to select from (null: the batch's own count)
cudaError_t launch_topk(const Scratch& s, long long n, int k, long long index_base,
                        int64_t* out_topk, int sms, const unsigned* count, cudaStream_t st);
// the k best of m (score, global index) pairs (cross-rank merge)
cudaError_t launch_merge_topk(const float* scores, const int64_t* idx, long long m, int k, int64_t* out,
                              cudaStream_t st);
cudaError_t launch_accumulate(StreamState* ss, const SelectState* st_, long long n_batch,
                              unsigned target, cudaStream_t st);
cudaError_t launch_stream_stats(const StreamState* ss, int64_t* out_stats, cudaStream_t st);

// sa.cu (explorer proposal step)
cudaError_t launch_sa_propose(const DecodeParams& dec, long long space, const int64_t* parent,
                              const uint32_t* knob_draw, const uint32_t* digit_draw, long long m,
                              long long* prop, unsigned* err, cudaStream_t st);
cudaError_t launch_sa_accept(long long space, const int64_t* parent, const float* parent_score,
                             const long long* prop, const float* perf, const float* log_u, long long m,
                             float temperature, int64_t* out_next, float* out_next_score,
                             int32_t* out_accepted, cudaStream_t st);

// screen_small.cu: the whole screening step in one launch for small batches
// (full V and P tables of the same depth held in shared memory together)
constexpr int kSmallMaxN = 8192;                 // candidates (keys the last CTA sorts)
constexpr size_t kSmallTableBytes = 160 * 1024;  // V + P tables
struct SmallPlan {
  int threads = 0;  // candidates per CTA (0: not eligible)
  int groups = 0;   // tree groups (CTA = 256 threads)
  size_t smem = 0;
  int ctas = 0;
};
SmallPlan plan_small(int F, long long n, const DeviceModel& V, const DeviceModel& P, int sms, int device_smem_optin);
cudaError_t launch_screen_small(const SmallPlan& pl, const DeviceModel& V, const DeviceModel& P, const float* feats,
                                int F, long long n, float tau, float* out_pvalid, float* out_perf, int64_t* out_topk,
                                int k, const Scratch& sc, int stall_cta, unsigned long long stall_ns,
                                cudaStream_t st);

// selftest.cu: a bounded wait that runs out (failure-detection self-test)
cudaError_t launch_wait_selftest(unsigned* err, unsigned long long limit_ns, cudaStream_t st);

// rerank.cu
cudaError_t launch_rerank(const DeviceModel& A, const float* feats, int F, long long n,
                          const int64_t* cand, int m, int n_final, float* out_score,
                          int64_t* out_final, unsigned long long* keys, unsigned* err,
                          cudaStream_t st);

}  // namespace mlt
