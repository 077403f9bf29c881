// Internal declarations shared by the libmlt translation units (not part of
// the C ABI).  Device table formats, launch descriptors and launchers.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

namespace mlt {

constexpr int kMaxKnobs = 16;
constexpr int kMaxOptions = 256;
constexpr int kMaxProgram = 256;
constexpr int kMaxF = 1024;
constexpr int kMaxK = 16384;
constexpr int kMaxDepth = 12;
constexpr int kMaxFullDepth = 10;  // deeper ensembles use the compact table

// Device error bits (accumulated in one word, read by mlt_sync_status).
constexpr unsigned kErrWaitTimeout = 1u;  // an mbarrier wait gave up
constexpr unsigned kErrSelect = 2u;       // top-k bookkeeping out of range

// A bounded device wait gives up after this many nanoseconds.
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

// ---------------------------------------------------------------------------
// Packed device tables
// ---------------------------------------------------------------------------
// Full table (depth D <= kMaxFullDepth): every tree is stored as a complete
// binary tree of depth D, `tree_bytes` apart (a multiple of 16):
//   I = 2^D - 1 internal records {float threshold; uint32 meta}, heap order,
//     meta bits 0..30 = feature index, bit 31 = NaN goes left;
//   L = 2^D leaf values (float), heap order of the last level.
// A shallower leaf is replicated into every leaf slot below it (its
// pass-through internal records test feature 0; any path gives the leaf).
//
// Compact table (any depth <= kMaxDepth): uint32 offsets[n_trees] (in
// records, from the start of the record area, which begins at byte
// align16(4 * n_trees)), then each tree's existing nodes in breadth-first
// order as {float value; uint32 meta}:
//   meta bit 30 = leaf (value = leaf output), bit 31 = NaN goes left,
//   bits 16..29 = index of the left child within the tree (right = left+1),
//   bits 0..15 = feature index.
enum TableKind : int { kTableFull = 0, kTableCompact = 1 };

constexpr uint32_t kMetaLeaf = 1u << 30;
constexpr uint32_t kMetaDefaultLeft = 1u << 31;

struct DeviceModel {
  const unsigned char* table = nullptr;
  size_t bytes = 0;
  int kind = kTableFull;
  int n_trees = 0;
  int depth = 0;
  uint32_t tree_bytes = 0;  // full tables
};

// ---------------------------------------------------------------------------
// Knob decoder (kernel parameter; ~5.3 KB)
// ---------------------------------------------------------------------------
struct DecodeParams {
  int n_knobs;
  int F;
  long long first_index;
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
constexpr int kRadixBins = 2048;  // 11-bit digits
constexpr int kRadixPasses = 6;   // 11+11+11+11+11+9 = 64 bits

struct SelectState {
  unsigned long long prefix;  // key bits fixed so far
  unsigned long long mask;    // which bits `prefix` fixes
  unsigned int remaining;     // rank still to find among prefix-matching keys
  unsigned int done;          // selection already determined
  unsigned int ticket;        // blocks finished in the current pass
  unsigned int n_sel;         // keys gathered
  unsigned int survivors;     // valid candidates of the current batch
  unsigned int k;             // requested k
  unsigned int hist[kRadixBins];
};

struct Scratch {
  uint32_t* masks = nullptr;         // [ceil(n/32)] validity ballots
  uint32_t* tile_counts = nullptr;   // [n_tiles] survivors per V tile
  uint32_t* tile_offsets = nullptr;  // [n_tiles] exclusive prefix
  uint32_t* rows = nullptr;          // [n] survivor positions, ascending
  unsigned long long* keys = nullptr;  // [n] (score, position) keys
  unsigned long long* sel = nullptr;   // [kMaxK] selected keys
  SelectState* state = nullptr;
  unsigned int* err = nullptr;       // device error word
};

// ---------------------------------------------------------------------------
// Launch descriptors
// ---------------------------------------------------------------------------
struct TraverseArgs {
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
  int max_depth;           // compact table
  float tau;
  // outputs
  float* out_pvalid;
  float* out_perf;
  uint32_t* masks;
  uint32_t* tile_counts;
  unsigned long long* keys;
  unsigned int* err;
  int decode;              // features built from candidate indices
};

struct ScreenShape {
  int threads;         // candidates per CTA
  size_t smem;         // dynamic shared memory bytes
  int chunk_trees;
  int nbuf;
  int group;           // trees walked together per thread (ILP)
};

// traverse.cu
ScreenShape plan_full(int F, int depth, int n_trees, uint32_t tree_bytes, int device_smem_optin);
ScreenShape plan_compact(int F, int device_smem_optin);
cudaError_t launch_traverse(const DeviceModel& m, const TraverseArgs& args, const DecodeParams* dec,
                            const ScreenShape& shape, long long n_tiles, cudaStream_t st);
cudaError_t launch_decode_rows(const DecodeParams& dec, long long n, uint8_t* out_knobs,
                               float* out_feats, cudaStream_t st);

// select.cu
cudaError_t launch_compact(const Scratch& s, long long n, int tile, long long n_tiles, int k,
                           cudaStream_t st);
cudaError_t launch_topk(const Scratch& s, long long n, int k, long long index_base,
                        int64_t* out_topk, cudaStream_t st);

}  // namespace mlt
