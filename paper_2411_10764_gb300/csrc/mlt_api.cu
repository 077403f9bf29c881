// libmlt C ABI: argument validation, ensemble packing, scratch management
// and the launch sequence of one screening pass (see include/mlt.h).
//
// ML^2Tuner (arXiv 2411.10764) Sec. 2: the explorer applies model V and
// model P to candidate configurations, discards those V predicts invalid and
// keeps the (alpha+1)N best by P.  One mlt_screen call = that step over a
// whole batch:
//   V pass (traverse.cu)  -> validity ballots, pvalid, -inf for the invalid
//   compaction (select.cu) -> ascending survivor list
//   P pass (traverse.cu)  -> P score per survivor + 64-bit rank keys
//   radix select + sort (select.cu) -> top-k indices
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "mlt.h"
#include <cuda_fp16.h>

#include "mlt_internal.cuh"
#include "peak.cuh"

// Scratch of mlt_screen_noalloc: one fixed array in the module's global
// memory (about 5.1 MB, held on every device that loads the library until
// the process exits), carved into the same pieces the allocating path uses.
namespace mlt_noalloc {
constexpr long long kMaxN = 262144;  // candidates per call
constexpr size_t align256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }
constexpr size_t kWords = kMaxN / 32 + 8;  // warp ballots; tile counters (tiles hold >= 32)
constexpr size_t kMasks = 0;
constexpr size_t kCounts = align256(kMasks + kWords * 4);
constexpr size_t kOffsets = align256(kCounts + kWords * 4);
constexpr size_t kRows = align256(kOffsets + kWords * 4);
constexpr size_t kKeys = align256(kRows + kMaxN * 4);
constexpr size_t kCand = align256(kKeys + kMaxN * 8);
constexpr size_t kState = align256(kCand + kMaxN * 8);
constexpr size_t kErr = align256(kState + sizeof(mlt::SelectState));
constexpr size_t kBytes = align256(kErr + sizeof(unsigned int));
constexpr int kMaxDevices = 64;
}  // namespace mlt_noalloc

static __device__ __align__(256) unsigned char g_noalloc_scratch[mlt_noalloc::kBytes];

namespace {

using namespace mlt;

thread_local std::string t_err;

constexpr long long kMaxMergePairs = 16LL * kMaxK;  // 16 ranks' top-k lists

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  t_err = buf;
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(MLT_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define MLT_CUDA(call, what)                      \
  do {                                            \
    cudaError_t e_ = (call);                      \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

struct Model {
  bool loaded = false;
  int device = -1;
  int F = 0;
  DeviceModel dm;
  unsigned char* owned = nullptr;
};

struct ScratchOwner {
  int device = -1;
  long long cap_n = -1;  // capacity in candidates
  Scratch s;
  void* block = nullptr;  // one allocation for everything sized by n
  SelectState* state = nullptr;
  unsigned int* err = nullptr;
  unsigned long long* rerank_keys = nullptr;  // [kMaxK]
  StreamState* stream = nullptr;              // batched accumulation
  // explorer proposal step buffers, grown with m
  long long sa_cap = -1;
  long long* sa_prop = nullptr;
  float* sa_pvalid = nullptr;
  float* sa_perf = nullptr;
  int64_t* sa_topk = nullptr;
  // rows of compiled-decoder batches, grown with n x F
  float* feat_buf = nullptr;
  long long feat_cap = 0;
  // host-buffer entry point staging
  long long host_cap_n = -1;
  int host_cap_F = 0;
  float* h_feats = nullptr;
  float* h_pvalid = nullptr;
  float* h_perf = nullptr;
  int64_t* h_topk = nullptr;
  // pipelined host batches: two staging sets, a copy stream and its events
  long long hb_cap_n = -1;
  int hb_cap_F = 0;
  float* hb_feats[2] = {nullptr, nullptr};
  float* hb_pvalid[2] = {nullptr, nullptr};
  float* hb_perf[2] = {nullptr, nullptr};
  int64_t* hb_topk[2] = {nullptr, nullptr};
  cudaStream_t hb_copy = nullptr;
  cudaEvent_t hb_in[2] = {nullptr, nullptr};    // batch's features are on the device
  cudaEvent_t hb_out[2] = {nullptr, nullptr};   // batch's screening is done
  cudaEvent_t hb_down[2] = {nullptr, nullptr};  // batch's results are on the host
};

std::mutex g_mu;
int g_F = 0;
long long g_launches = 0;

// Phase profiling: one set of 5 events per recorded screening call.
constexpr int kPhases = 4;
bool g_profile = false;
std::vector<cudaEvent_t> g_events;  // pool, 5 per call
size_t g_events_used = 0;
Model g_models[3];
ScratchOwner g_scr;
int g_optin = -1;
int g_sms = -1;
ShapeOverride g_shape[3];
// failure-detection self-test, armed by mlt_selftest_walk_timeout: the next
// full-table V pass makes CTA g_stall_cta wait on a barrier phase that
// nothing completes, for g_stall_ns (one shot)
int g_head_levels = kSplitHeadDefault;  // split tables for deep V and P models (0: compact tables)
long long g_small_max = kSmallMaxN;     // batches up to this size screen in one launch when eligible
// decoded batches of at least this many candidates use the compiled feature
// program (0: never); the count of calls that did
long long g_jit_min_n = kDecodeJitMinN;
long long g_jit_calls = 0;
int g_stall_cta = -1;
unsigned long long g_stall_ns = 0;

size_t align16(size_t v) { return (v + 15) & ~static_cast<size_t>(15); }

int current_device(int* dev) {
  MLT_CUDA(cudaGetDevice(dev), "cudaGetDevice");
  return MLT_OK;
}

int smem_optin() {
  if (g_optin < 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 48 * 1024;
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
      return 48 * 1024;
    g_optin = v;
  }
  return g_optin;
}

int sm_count() {
  if (g_sms < 0) {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return 1;
    g_sms = v;
  }
  return g_sms;
}

void free_model(Model& m) {
  if (m.owned != nullptr) {
    cudaDeviceSynchronize();  // queued screens may still read the table
    cudaFree(m.owned);
  }
  m = Model();
}

// Scratch sized by n candidates (plus the fixed pieces).
// The compiled decoder's row buffer: at least `elems` floats on the scratch
// device (grown, never shrunk; kept until exit).  False when it cannot be
// had (the caller then decodes inside the walks, which needs no buffer).
bool try_feat_buf(long long elems) {
  if (elems <= g_scr.feat_cap) return true;
  if (g_scr.feat_buf != nullptr) {
    cudaDeviceSynchronize();
    cudaFree(g_scr.feat_buf);
    g_scr.feat_buf = nullptr;
    g_scr.feat_cap = 0;
  }
  void* p = nullptr;
  if (cudaMalloc(&p, static_cast<size_t>(elems) * sizeof(float)) != cudaSuccess) {
    cudaGetLastError();  // clear the allocation failure
    return false;
  }
  g_scr.feat_buf = static_cast<float*>(p);
  g_scr.feat_cap = elems;
  return true;
}

int ensure_scratch(long long n) {
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  if (g_scr.err == nullptr || g_scr.device != dev) {
    if (g_scr.device != -1 && g_scr.device != dev)
      return fail(MLT_EINVAL, "libmlt scratch lives on device %d, current device is %d", g_scr.device, dev);
    MLT_CUDA(cudaMalloc(&g_scr.err, sizeof(unsigned int)), "cudaMalloc(error word)");
    MLT_CUDA(cudaMemset(g_scr.err, 0, sizeof(unsigned int)), "cudaMemset(error word)");
    MLT_CUDA(cudaMalloc(&g_scr.state, sizeof(SelectState)), "cudaMalloc(select state)");
    MLT_CUDA(cudaMemset(g_scr.state, 0, sizeof(SelectState)), "cudaMemset(select state)");
    MLT_CUDA(cudaMalloc(&g_scr.rerank_keys, sizeof(unsigned long long) * kMaxK), "cudaMalloc(rerank keys)");
    MLT_CUDA(cudaMalloc(&g_scr.stream, sizeof(StreamState)), "cudaMalloc(stream state)");
    g_scr.device = dev;
  }
  if (n > g_scr.cap_n) {
    long long cap = n < 1024 ? 1024 : n;
    const long long words = (cap + 31) / 32 + 8;
    const size_t b_masks = align16(words * 4);
    const size_t b_tiles = align16(words * 4);  // tiles are >= 32 candidates
    const size_t b_rows = align16(cap * 4);
    const size_t b_keys = align16(cap * 8);
    const size_t total = b_masks + 2 * b_tiles + b_rows + 2 * b_keys;
    if (g_scr.block != nullptr) {
      cudaDeviceSynchronize();
      cudaFree(g_scr.block);
      g_scr.block = nullptr;
      g_scr.cap_n = -1;
    }
    void* blk = nullptr;
    cudaError_t e = cudaMalloc(&blk, total);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(MLT_ENOMEM, "cannot allocate %zu bytes of screening scratch", total);
    }
    unsigned char* p = static_cast<unsigned char*>(blk);
    g_scr.s.masks = reinterpret_cast<uint32_t*>(p);
    p += b_masks;
    g_scr.s.tile_counts = reinterpret_cast<uint32_t*>(p);
    p += b_tiles;
    g_scr.s.tile_offsets = reinterpret_cast<uint32_t*>(p);
    p += b_tiles;
    g_scr.s.rows = reinterpret_cast<uint32_t*>(p);
    p += b_rows;
    g_scr.s.keys = reinterpret_cast<unsigned long long*>(p);
    p += b_keys;
    g_scr.s.cand = reinterpret_cast<unsigned long long*>(p);
    g_scr.block = blk;
    g_scr.cap_n = cap;
  }
  g_scr.s.state = g_scr.state;
  g_scr.s.err = g_scr.err;
  return MLT_OK;
}

// sigmoid(m) >= thr  <=>  thr * (1 + e^-m) <= 1  <=>  thr * expm1(-m) <= 1 - 2 thr
bool cut_passes(float m, float thr) {
  const long double lhs = static_cast<long double>(thr) * expm1l(-static_cast<long double>(m));
  const long double rhs = 1.0L - 2.0L * static_cast<long double>(thr);
  return lhs <= rhs;
}

float validity_cut(float thr) {
  float m = static_cast<float>(std::log(static_cast<double>(thr) / (1.0 - static_cast<double>(thr))));
  if (!cut_passes(m, thr)) {
    while (!cut_passes(m, thr)) m = std::nextafterf(m, INFINITY);
  } else {
    for (;;) {
      const float d = std::nextafterf(m, -INFINITY);
      if (!cut_passes(d, thr)) break;
      m = d;
    }
  }
  return m == 0.0f ? 0.0f : m;
}

int check_screen_args(long long n, float thr, int k) {
  if (n < 0 || n > 0x7FFFFFFFLL) return fail(MLT_EINVAL, "n must lie in [0, 2^31-1], got %lld", n);
  if (!(thr > 0.0f && thr < 1.0f)) return fail(MLT_EINVAL, "thr must lie in (0, 1)");
  if (k < 1 || k > kMaxK) return fail(MLT_EINVAL, "k must lie in [1, %d], got %d", kMaxK, k);
  return MLT_OK;
}

// decoded: the features are built from candidate indices (half tables need
// a stored feature matrix).
int check_models(int dev, bool decoded = false) {
  for (int id : {MLT_MODEL_V, MLT_MODEL_P}) {
    const Model& m = g_models[id];
    if (!m.loaded) return fail(MLT_ENOMODEL, "model %s is not loaded", id == 0 ? "V" : "P");
    if (m.F != g_F) return fail(MLT_ENOMODEL, "model %s was loaded for F=%d, current F=%d", id == 0 ? "V" : "P", m.F, g_F);
    if (m.device != dev) return fail(MLT_EINVAL, "model %s lives on device %d, current device is %d", id == 0 ? "V" : "P", m.device, dev);
    if (decoded && m.dm.kind == kTableHalf)
      return fail(MLT_EINVAL, "model %s has half tables, which need stored features", id == 0 ? "V" : "P");
  }
  return MLT_OK;
}

// v_pass: n_eff is the exact number of candidates; otherwise it is an
// estimate of the survivors.  Full-table tiles are balanced over the SMs.
ScreenShape plan_for(const DeviceModel& dm, int F, long long n_eff, const ShapeOverride& ov, bool v_pass) {
  const bool half = dm.kind == kTableHalf;
  ScreenShape s = dm.kind == kTableCompact ? plan_compact(F, n_eff, sm_count(), smem_optin(), ov)
                  : dm.kind == kTableSplit
                      ? plan_split(F, dm.n_trees, dm.tree_bytes, n_eff, sm_count(), smem_optin(), ov)
                      : plan_full(F, dm.n_trees, dm.tree_bytes, n_eff, sm_count(), smem_optin(), ov, half);
  if (s.threads == 0 && (ov.threads || ov.chunk_trees || ov.nbuf || ov.lanes || ov.group))
    return plan_for(dm, F, n_eff, ShapeOverride(), v_pass);
  // no more CTAs per SM than the plan counted on
  if (dm.kind != kTableCompact) s = cap_residency(s, smem_optin());
  return s;
}

int build_decoder(const int32_t* radices, const float* option_values, int n_knobs,
                  const mlt_feat_op* program, int F, long long first_index, long long n,
                  DecodeParams* d) {
  if (radices == nullptr || option_values == nullptr || program == nullptr)
    return fail(MLT_EINVAL, "radices, option_values and program must be non-NULL");
  if (n_knobs < 1 || n_knobs > kMaxKnobs) return fail(MLT_EINVAL, "n_knobs must lie in [1, %d]", kMaxKnobs);
  if (F < 1 || F > kMaxProgram) return fail(MLT_EINVAL, "program length must lie in [1, %d]", kMaxProgram);
  if (first_index < 0 || n < 0) return fail(MLT_EINVAL, "first_index and n must be non-negative");
  std::memset(d, 0, sizeof(*d));
  d->n_knobs = n_knobs;
  d->F = F;
  d->first_index = first_index;
  int off = 0;
  long double space = 1.0L;
  for (int j = 0; j < n_knobs; ++j) {
    if (radices[j] < 1 || radices[j] > 256) return fail(MLT_EINVAL, "radix %d of knob %d outside [1, 256]", radices[j], j);
    d->radix[j] = radices[j];
    d->opt_off[j] = off;
    off += radices[j];
    if (off > kMaxOptions) return fail(MLT_EINVAL, "more than %d option values in total", kMaxOptions);
    space *= radices[j];
  }
  if (static_cast<long double>(first_index) + static_cast<long double>(n) > space)
    return fail(MLT_EINVAL, "candidates past the end of the knob space");
  std::memcpy(d->opts, option_values, sizeof(float) * off);
  for (int f = 0; f < F; ++f) {
    const mlt_feat_op& o = program[f];
    if (o.op < 0 || o.op > MLT_OP_EQ) return fail(MLT_EINVAL, "feature %d: unknown opcode %d", f, o.op);
    if (o.a < -1 || o.a >= n_knobs + f || o.b < -1 || o.b >= n_knobs + f)
      return fail(MLT_EINVAL, "feature %d: operand refers to an unknown slot", f);
    d->op[f] = o.op;
    d->a[f] = o.a;
    d->b[f] = o.b;
    d->c[f] = o.c;
  }
  return MLT_OK;
}

// Validate the heap-order ensemble and pack it for the device.
int pack_ensemble(const mlt_node* nodes, int n_trees, int depth, int F, std::vector<unsigned char>& out,
                  DeviceModel& dm) {
  const int slots = (2 << depth) - 1;
  std::vector<unsigned char> reach(slots);
  std::vector<int> depth_of(slots);
  for (int j = 0; j < slots; ++j) depth_of[j] = 31 - __builtin_clz(static_cast<unsigned>(j + 1));
  long double leaf_bound = 0.0L;
  for (int t = 0; t < n_trees; ++t) {
    const mlt_node* tr = nodes + static_cast<size_t>(t) * slots;
    std::fill(reach.begin(), reach.end(), 0);
    reach[0] = 1;
    float maxabs = 0.0f;
    for (int j = 0; j < slots; ++j) {
      if (!reach[j]) continue;
      const mlt_node& nd = tr[j];
      if (nd.feature == -2) return fail(MLT_EINVAL, "tree %d slot %d: reachable slot is unused", t, j);
      if (nd.feature < -2) return fail(MLT_EINVAL, "tree %d slot %d: bad feature code %d", t, j, nd.feature);
      if (!std::isfinite(nd.value)) return fail(MLT_EINVAL, "tree %d slot %d: value is not finite", t, j);
      if (nd.feature == -1) {
        maxabs = std::fmax(maxabs, std::fabs(nd.value));
        continue;
      }
      if (depth_of[j] >= depth) return fail(MLT_EINVAL, "tree %d slot %d: split below the depth limit", t, j);
      if (nd.feature >= F) return fail(MLT_EINVAL, "tree %d slot %d: feature %d >= F=%d", t, j, nd.feature, F);
      reach[2 * j + 1] = 1;
      reach[2 * j + 2] = 1;
    }
    leaf_bound += maxabs;
  }
  if (leaf_bound >= 1e37L) return fail(MLT_EINVAL, "leaf magnitudes could overflow the fp32 sum");

  dm.n_trees = n_trees;
  dm.depth = depth;
  if (depth <= kMaxFullDepth) {
    const FullLayout lay = full_layout(depth);
    const size_t tb = lay.bytes;
    dm.kind = kTableFull;
    dm.tree_bytes = lay.bytes;
    out.assign(tb * n_trees, 0);
    const int inner = (1 << depth) - 1;  // internal heap slots of the complete tree
    std::vector<float> inherit(slots);
    std::vector<float> thr_of(inner);
    std::vector<uint32_t> meta_of(inner);
    for (int t = 0; t < n_trees; ++t) {
      const mlt_node* tr = nodes + static_cast<size_t>(t) * slots;
      unsigned char* dst = out.data() + tb * t;
      std::fill(reach.begin(), reach.end(), 0);
      reach[0] = 1;
      for (int j = 0; j < slots; ++j) {
        const mlt_node& nd = tr[j];
        const bool split = reach[j] && nd.feature >= 0;
        if (split) {
          reach[2 * j + 1] = 1;
          reach[2 * j + 2] = 1;
        }
        if (reach[j] && nd.feature == -1)
          inherit[j] = nd.value;
        else if (!reach[j])
          inherit[j] = inherit[(j - 1) / 2];  // below a leaf: copy it down
        else
          inherit[j] = 0.0f;
        if (j < inner) {
          thr_of[j] = split ? nd.value : 0.0f;
          meta_of[j] = split ? (static_cast<uint32_t>(nd.feature) | (nd.default_left ? kMetaDefaultLeft : 0u)) : 0u;
        }
      }
      for (uint32_t j = 0; j < static_cast<uint32_t>(inner); ++j) {
        if (j < lay.n_top) {
          std::memcpy(dst + 8 * j, &thr_of[j], 4);
          std::memcpy(dst + 8 * j + 4, &meta_of[j], 4);
        } else {
          // feature (< kMaxF) in bits 0..14, the NaN-left flag in bit 15
          const uint16_t m = static_cast<uint16_t>((meta_of[j] & kMeta16Feature) |
                                                   ((meta_of[j] & kMetaDefaultLeft) ? kMeta16Left : 0u));
          std::memcpy(dst + lay.off_thr + 4 * (j - lay.n_top), &thr_of[j], 4);
          std::memcpy(dst + lay.off_meta + 2 * (j - lay.n_top), &m, 2);
        }
      }
      // the leaf below each path: child heap index c of a last-level node
      for (uint32_t c = static_cast<uint32_t>(inner); c < static_cast<uint32_t>(slots); ++c) {
        const float v = inherit[c];
        std::memcpy(dst + lay.off_leaf + 4 * (c - inner), &v, 4);
      }
    }
  } else {
    dm.kind = kTableCompact;
    dm.tree_bytes = 0;
    std::vector<uint32_t> offsets(n_trees);
    std::vector<uint32_t> recs;
    std::vector<int> order;
    for (int t = 0; t < n_trees; ++t) {
      const mlt_node* tr = nodes + static_cast<size_t>(t) * slots;
      offsets[t] = static_cast<uint32_t>(recs.size() / 2);
      order.assign(1, 0);
      for (size_t q = 0; q < order.size(); ++q) {
        const mlt_node& nd = tr[order[q]];
        float v = nd.value;
        uint32_t meta;
        if (nd.feature >= 0) {
          const uint32_t left = static_cast<uint32_t>(order.size());
          if (left > kCompactChildMask) return fail(MLT_EINVAL, "tree %d has too many nodes", t);
          order.push_back(2 * order[q] + 1);
          order.push_back(2 * order[q] + 2);
          meta = static_cast<uint32_t>(nd.feature) | (left << kCompactChildShift) |
                 (nd.default_left ? kMetaDefaultLeft : 0u);
        } else {
          meta = kMetaLeaf;
        }
        uint32_t vb;
        std::memcpy(&vb, &v, 4);
        recs.push_back(vb);
        recs.push_back(meta);
      }
    }
    const size_t head = align16(static_cast<size_t>(n_trees) * 4);
    out.assign(head + recs.size() * 4, 0);
    std::memcpy(out.data(), offsets.data(), offsets.size() * 4);
    std::memcpy(out.data() + head, recs.data(), recs.size() * 4);
  }
  return MLT_OK;
}

// The whole screening sequence on `st` with scratch `s` (caller holds g_mu).
// `profile_ok`: phase events may be recorded.
int run_screen_with(cudaStream_t st, const float* feats, const DecodeParams* dec, long long n, float thr,
                    int k, float* out_pvalid, float* out_perf, int64_t* out_topk, const Scratch& s,
                    bool profile_ok) {
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  rc = check_models(dev, dec != nullptr);
  if (rc != MLT_OK) return rc;
  const DeviceModel& V = g_models[MLT_MODEL_V].dm;
  const DeviceModel& P = g_models[MLT_MODEL_P].dm;
  // a large decoded batch: the compiled feature program writes its rows
  // once, and the walks stage them like stored features (the same bits as
  // decoding inside the walks); top-k positions stay candidate indices
  const long long topk_base = dec ? dec->first_index : 0;
  const DecodeParams* jit_dec = nullptr;
  JitDecoder jd{};
  if (dec != nullptr && g_jit_min_n > 0 && n >= g_jit_min_n) {
    jd = jit_decoder_for(*dec, dev);
    if (jd.fn != nullptr && try_feat_buf(n * static_cast<long long>(g_F))) {
      jit_dec = dec;
      feats = g_scr.feat_buf;
      dec = nullptr;
    }
  }
  // the P pass walks the survivors; plan it for about half the batch
  const ScreenShape sv = plan_for(V, g_F, n, g_shape[MLT_MODEL_V], true);
  const ScreenShape sp = plan_for(P, g_F, (n + 1) / 2, g_shape[MLT_MODEL_P], false);
  if (sv.threads == 0 || sp.threads == 0) return fail(MLT_EINVAL, "F=%d leaves no room for a shared-memory tile", g_F);
  TraverseArgs a{};
  a.feats = feats;
  a.F = g_F;
  a.n = n;
  a.vec4 = (feats != nullptr && (reinterpret_cast<uintptr_t>(feats) & 15u) == 0 && (g_F & 3) == 0) ? 1 : 0;
  a.state = s.state;
  a.rows = s.rows;
  a.tau = validity_cut(thr);
  a.out_pvalid = out_pvalid;
  a.out_perf = out_perf;
  a.masks = s.masks;
  a.tile_counts = s.tile_counts;
  a.keys = s.keys;
  a.hist = s.state->hist;
  a.tile_offsets = s.tile_offsets;
  a.state_rw = s.state;
  a.err = s.err;
  a.decode = dec != nullptr;

  TraverseArgs av = a;
  av.p_pass = 0;
  av.table = V.table;
  av.n_trees = V.n_trees;
  av.tree_bytes = V.tree_bytes;
  av.chunk_trees = sv.chunk_trees;
  av.nbuf = sv.nbuf;
  av.max_depth = V.depth;
  av.tail = reinterpret_cast<const uint2*>(V.tail);
  // every call starts from a fresh selection state: its tickets decide which
  // CTA scans the tile counts and ranks the keys, so a count left behind by
  // an earlier call (one that stopped part-way) must not carry over
  MLT_CUDA(cudaMemsetAsync(s.state, 0, sizeof(SelectState), st), "reset selection state");
  cudaEvent_t* ev = nullptr;
  if (g_profile && profile_ok) {
    if (g_events_used + kPhases + 1 > g_events.size()) {
      for (int i = 0; i <= kPhases; ++i) {
        cudaEvent_t e;
        MLT_CUDA(cudaEventCreate(&e), "cudaEventCreate");
        g_events.push_back(e);
      }
    }
    ev = &g_events[g_events_used];
    g_events_used += kPhases + 1;
    MLT_CUDA(cudaEventRecord(ev[0], st), "cudaEventRecord");
  }
  if (jit_dec != nullptr) {  // recorded with the V phase
    MLT_CUDA(launch_jit_decode(jd, *jit_dec, n, g_scr.feat_buf, st), "compiled decoder launch");
    g_launches += 1;
    g_jit_calls += 1;
  }
  // a small batch of stored features: the whole step in one launch (its
  // time is recorded as the V phase)
  if (dec == nullptr && jit_dec == nullptr && n <= g_small_max) {
    const SmallPlan pl = plan_small(g_F, n, V, P, sm_count(), smem_optin());
    if (pl.threads > 0) {
      int stall = -1;
      unsigned long long stall_ns = 0;
      if (g_stall_cta >= 0) {
        stall = static_cast<int>(std::min<long long>(g_stall_cta, pl.ctas - 1));
        stall_ns = g_stall_ns;
        g_stall_cta = -1;
      }
      MLT_CUDA(launch_screen_small(pl, V, P, feats, g_F, n, a.tau, out_pvalid, out_perf, out_topk, k, s, stall,
                                   stall_ns, st),
               "small-batch screening launch");
      if (ev)
        for (int i = 1; i <= kPhases; ++i) MLT_CUDA(cudaEventRecord(ev[i], st), "cudaEventRecord");
      g_launches += 1;
      return MLT_OK;
    }
  }
  const long long tiles_v = (n + sv.threads - 1) / sv.threads;
  if (g_stall_cta >= 0 && V.kind != kTableCompact && tiles_v > 0) {
    av.stall_cta = static_cast<int>(std::min<long long>(g_stall_cta, tiles_v - 1));
    av.stall_ns = g_stall_ns;
    g_stall_cta = -1;
  }
  MLT_CUDA(dec ? launch_traverse_dec(V, av, *dec, sv, tiles_v, st) : launch_traverse(V, av, sv, tiles_v, st),
           "V pass launch");
  if (ev) MLT_CUDA(cudaEventRecord(ev[1], st), "cudaEventRecord");
  MLT_CUDA(launch_compact(s, n, sv.threads, tiles_v, nullptr, st), "compaction launch");
  if (ev) MLT_CUDA(cudaEventRecord(ev[2], st), "cudaEventRecord");

  TraverseArgs ap = a;
  ap.p_pass = 1;
  ap.table = P.table;
  ap.n_trees = P.n_trees;
  ap.tree_bytes = P.tree_bytes;
  ap.chunk_trees = sp.chunk_trees;
  ap.nbuf = sp.nbuf;
  ap.max_depth = P.depth;
  ap.tail = reinterpret_cast<const uint2*>(P.tail);
  const long long tiles_p = (n + sp.threads - 1) / sp.threads;
  MLT_CUDA(dec ? launch_traverse_dec(P, ap, *dec, sp, tiles_p, st) : launch_traverse(P, ap, sp, tiles_p, st),
           "P pass launch");
  if (ev) MLT_CUDA(cudaEventRecord(ev[3], st), "cudaEventRecord");
  MLT_CUDA(launch_topk(s, n, k, topk_base, out_topk, sm_count(), nullptr, st), "top-k launch");
  if (ev) MLT_CUDA(cudaEventRecord(ev[4], st), "cudaEventRecord");
  g_launches += (tiles_v > 0 ? 1 : 0) + (tiles_v > 0 ? 1 : 0) + (tiles_p > 0 ? 1 : 0) + 1;
  return MLT_OK;
}

// Device address of g_noalloc_scratch on the current device, resolved the
// first time per device (in host code the array's name is only a stand-in).
unsigned char* g_noalloc_base[mlt_noalloc::kMaxDevices] = {};

int noalloc_scratch(int dev, Scratch* out) {
  using namespace mlt_noalloc;
  if (dev < 0 || dev >= kMaxDevices) return fail(MLT_EINVAL, "device %d out of range for the static scratch", dev);
  if (g_noalloc_base[dev] == nullptr) {
    void* p = nullptr;
    MLT_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch), "cudaGetSymbolAddress(static scratch)");
    // the error word starts at zero (it is cleared again whenever
    // mlt_sync_status reads it)
    MLT_CUDA(cudaMemset(static_cast<unsigned char*>(p) + kErr, 0, sizeof(unsigned int)),
             "clear static error word");
    g_noalloc_base[dev] = static_cast<unsigned char*>(p);
  }
  unsigned char* b = g_noalloc_base[dev];
  out->masks = reinterpret_cast<uint32_t*>(b + kMasks);
  out->tile_counts = reinterpret_cast<uint32_t*>(b + kCounts);
  out->tile_offsets = reinterpret_cast<uint32_t*>(b + kOffsets);
  out->rows = reinterpret_cast<uint32_t*>(b + kRows);
  out->keys = reinterpret_cast<unsigned long long*>(b + kKeys);
  out->cand = reinterpret_cast<unsigned long long*>(b + kCand);
  out->state = reinterpret_cast<SelectState*>(b + kState);
  out->err = reinterpret_cast<unsigned int*>(b + kErr);
  return MLT_OK;
}

// Batched accumulation (ML^2Tuner Sec. 2: the explorer applies P and V
// until (alpha+1)N configurations have accumulated): batches of `batch`
// candidates are all enqueued; after each, a one-thread kernel adds the
// batch's survivors to the running count and raises a device flag once it
// reaches `target`, which makes every later batch's kernels return at once.
// One top-k then ranks all survivors kept.  The result equals screening the
// consumed prefix of the candidates as a single batch.
int run_stream(cudaStream_t st, const float* feats, const DecodeParams* dec0, long long n_total, long long batch,
               long long target, float thr, int k, float* out_pvalid, float* out_perf, int64_t* out_topk,
               int64_t* out_stats) {
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  rc = check_models(dev, dec0 != nullptr);
  if (rc != MLT_OK) return rc;
  rc = ensure_scratch(n_total);  // every kept survivor's key fits
  if (rc != MLT_OK) return rc;
  const Scratch& s = g_scr.s;
  StreamState* ss = g_scr.stream;
  const DeviceModel& V = g_models[MLT_MODEL_V].dm;
  const DeviceModel& P = g_models[MLT_MODEL_P].dm;
  const long long per = std::min(batch, std::max(1LL, n_total));
  const ScreenShape sv = plan_for(V, g_F, per, g_shape[MLT_MODEL_V], true);
  const ScreenShape sp = plan_for(P, g_F, (per + 1) / 2, g_shape[MLT_MODEL_P], false);
  if (sv.threads == 0 || sp.threads == 0) return fail(MLT_EINVAL, "F=%d leaves no room for a shared-memory tile", g_F);
  MLT_CUDA(cudaMemsetAsync(s.state, 0, sizeof(SelectState), st), "reset selection state");
  MLT_CUDA(cudaMemsetAsync(ss, 0, sizeof(StreamState), st), "reset stream state");
  const unsigned tgt = static_cast<unsigned>(std::min<long long>(target, 0xFFFFFFFFLL));
  TraverseArgs a{};
  a.F = g_F;
  a.state = s.state;
  a.rows = s.rows;
  a.tau = validity_cut(thr);
  a.masks = s.masks;
  a.tile_counts = s.tile_counts;
  a.keys = s.keys;
  a.hist = s.state->hist;
  a.tile_offsets = s.tile_offsets;
  a.state_rw = s.state;
  a.err = s.err;
  a.decode = dec0 != nullptr;
  a.stream = ss;
  long long launches = 0;
  for (long long b0 = 0; b0 < n_total; b0 += batch) {
    const long long nb = std::min(batch, n_total - b0);
    TraverseArgs ab = a;
    ab.n = nb;
    ab.pos_base = b0;
    ab.feats = feats ? feats + b0 * g_F : nullptr;
    ab.vec4 = (ab.feats != nullptr && (reinterpret_cast<uintptr_t>(ab.feats) & 15u) == 0 && (g_F & 3) == 0) ? 1 : 0;
    ab.out_pvalid = out_pvalid ? out_pvalid + b0 : nullptr;
    ab.out_perf = out_perf ? out_perf + b0 : nullptr;
    DecodeParams d;
    if (dec0) {
      d = *dec0;
      d.first_index += b0;
    }
    TraverseArgs av = ab;
    av.p_pass = 0;
    av.table = V.table;
    av.n_trees = V.n_trees;
    av.tree_bytes = V.tree_bytes;
    av.chunk_trees = sv.chunk_trees;
    av.nbuf = sv.nbuf;
    av.max_depth = V.depth;
    av.tail = reinterpret_cast<const uint2*>(V.tail);
    const long long tiles_v = (nb + sv.threads - 1) / sv.threads;
    MLT_CUDA(dec0 ? launch_traverse_dec(V, av, d, sv, tiles_v, st) : launch_traverse(V, av, sv, tiles_v, st),
             "V pass launch");
    MLT_CUDA(launch_compact(s, nb, sv.threads, tiles_v, ss, st), "compaction launch");
    TraverseArgs ap = ab;
    ap.p_pass = 1;
    ap.table = P.table;
    ap.n_trees = P.n_trees;
    ap.tree_bytes = P.tree_bytes;
    ap.chunk_trees = sp.chunk_trees;
    ap.nbuf = sp.nbuf;
    ap.max_depth = P.depth;
    ap.tail = reinterpret_cast<const uint2*>(P.tail);
    const long long tiles_p = (nb + sp.threads - 1) / sp.threads;
    MLT_CUDA(dec0 ? launch_traverse_dec(P, ap, d, sp, tiles_p, st) : launch_traverse(P, ap, sp, tiles_p, st),
             "P pass launch");
    MLT_CUDA(launch_accumulate(ss, s.state, nb, tgt, st), "accumulate launch");
    launches += 4;
  }
  MLT_CUDA(launch_topk(s, n_total, k, dec0 ? dec0->first_index : 0, out_topk, sm_count(), &ss->total, st),
           "top-k launch");
  launches += 1;
  if (out_stats) {
    MLT_CUDA(launch_stream_stats(ss, out_stats, st), "stats launch");
    launches += 1;
  }
  g_launches += launches;
  return MLT_OK;
}

int check_stream_args(long long n_total, long long batch, long long target, float thr, int k) {
  int rc = check_screen_args(n_total, thr, k);
  if (rc != MLT_OK) return rc;
  if (batch < 1) return fail(MLT_EINVAL, "batch must be >= 1");
  if (target < 1) return fail(MLT_EINVAL, "target must be >= 1");
  if ((n_total + batch - 1) / batch > 65536) return fail(MLT_EINVAL, "more than 65536 batches");
  return MLT_OK;
}

// The screening sequence with the library's own (allocated) scratch.
int run_screen(cudaStream_t st, const float* feats, const DecodeParams* dec, long long n, float thr, int k,
               float* out_pvalid, float* out_perf, int64_t* out_topk) {
  const int rc = ensure_scratch(n);
  if (rc != MLT_OK) return rc;
  return run_screen_with(st, feats, dec, n, thr, k, out_pvalid, out_perf, out_topk, g_scr.s, true);
}

// Split table (kTableSplit, deep models V and P): validate like
// pack_ensemble, then store each tree's first H levels and its level-H exits
// as a head block and everything below level H as breadth-first compact
// records in one tail array (layout in mlt_internal.cuh).
int pack_split(const mlt_node* nodes, int n_trees, int depth, int F, int H, std::vector<unsigned char>& out,
               DeviceModel& dm) {
  {
    std::vector<unsigned char> scratch;
    DeviceModel probe;
    const int rc = pack_ensemble(nodes, n_trees, depth, F, scratch, probe);  // validation
    if (rc != MLT_OK) return rc;
  }
  const int slots = (2 << depth) - 1;
  const uint32_t hb = split_head_bytes(H);
  const int n_head = (1 << H) - 1;         // slots of levels 0 .. H-1
  const int n_exit_end = (2 << H) - 1;     // level-H slots end here
  const size_t tail_off = align16(static_cast<size_t>(n_trees) * hb);
  std::vector<unsigned char> heads(tail_off, 0);
  std::vector<uint32_t> recs;  // tail records, two words each
  std::vector<unsigned char> reach(slots);
  std::vector<float> inherit(n_exit_end);
  std::vector<int> order;
  // every node sends a missing value right: a node whose missing values go
  // left is stored with its subtrees swapped, the negate bit (31) set and
  // threshold -prev(t), so that "x < t or x missing" (its old left side) is
  // "-x >= -prev(t) or -x missing" (its new right side)
  std::vector<mlt_node> tn(slots);
  std::vector<unsigned char> neg(slots);
  std::vector<std::pair<int, int>> stack;
  auto split_meta = [&](int j, uint32_t left) {
    return static_cast<uint32_t>(tn[j].feature) | (left << kCompactChildShift) | (neg[j] ? kMetaDefaultLeft : 0u);
  };
  for (int t = 0; t < n_trees; ++t) {
    const mlt_node* orig = nodes + static_cast<size_t>(t) * slots;
    for (mlt_node& nd : tn) nd = mlt_node{-2, 0.0f, 0, {0, 0, 0}};
    std::fill(neg.begin(), neg.end(), 0);
    stack.assign(1, {0, 0});
    while (!stack.empty()) {
      const auto [j, jn] = stack.back();
      stack.pop_back();
      const mlt_node& nd = orig[j];
      tn[jn] = nd;
      if (nd.feature < 0) continue;
      if (nd.default_left) {
        tn[jn].value = -std::nextafterf(nd.value, -INFINITY);
        neg[jn] = 1;
        stack.push_back({2 * j + 1, 2 * jn + 2});
        stack.push_back({2 * j + 2, 2 * jn + 1});
      } else {
        stack.push_back({2 * j + 1, 2 * jn + 1});
        stack.push_back({2 * j + 2, 2 * jn + 2});
      }
    }
    const mlt_node* tr = tn.data();
    unsigned char* dst = heads.data() + static_cast<size_t>(t) * hb;
    std::fill(reach.begin(), reach.end(), 0);
    reach[0] = 1;
    for (int j = 0; j < slots; ++j) {
      if (reach[j] && tr[j].feature >= 0) {
        reach[2 * j + 1] = 1;
        reach[2 * j + 2] = 1;
      }
    }
    for (int j = 0; j < n_exit_end; ++j) {
      if (reach[j] && tr[j].feature == -1)
        inherit[j] = tr[j].value;
      else if (!reach[j])
        inherit[j] = inherit[(j - 1) / 2];  // below a leaf: copy it down
      else
        inherit[j] = 0.0f;
    }
    // levels 0 .. H-1: splits, or pass-through records
    for (int j = 0; j < n_head; ++j) {
      const mlt_node& nd = tr[j];
      const bool split = reach[j] && nd.feature >= 0;
      const float thr = split ? nd.value : 0.0f;
      const uint32_t meta = split ? (static_cast<uint32_t>(nd.feature) | (neg[j] ? kMetaDefaultLeft : 0u)) : 0u;
      std::memcpy(dst + 8 * j, &thr, 4);
      std::memcpy(dst + 8 * j + 4, &meta, 4);
    }
    // level H: leaves, or split nodes whose children open the tail
    const size_t base = recs.size() / 2;
    if (base > 0xFFFFFFFFull) return fail(MLT_EINVAL, "split table too large");
    order.clear();
    for (int j = n_head; j < n_exit_end; ++j) {
      const mlt_node& nd = tr[j];
      float v;
      uint32_t meta;
      if (reach[j] && nd.feature >= 0) {
        const uint32_t left = static_cast<uint32_t>(order.size());
        order.push_back(2 * j + 1);
        order.push_back(2 * j + 2);
        v = nd.value;
        meta = split_meta(j, left);
      } else {
        v = inherit[j];
        meta = kMetaLeaf;
      }
      std::memcpy(dst + 8 * j, &v, 4);
      std::memcpy(dst + 8 * j + 4, &meta, 4);
    }
    const uint32_t b32 = static_cast<uint32_t>(base);
    std::memcpy(dst + hb - 8, &b32, 4);
    // below level H, breadth first (children adjacent)
    for (size_t q = 0; q < order.size(); ++q) {
      const mlt_node& nd = tr[order[q]];
      uint32_t vb, meta;
      std::memcpy(&vb, &nd.value, 4);
      if (nd.feature >= 0) {
        const uint32_t left = static_cast<uint32_t>(order.size());
        if (left > kCompactChildMask) return fail(MLT_EINVAL, "tree %d has too many nodes", t);
        order.push_back(2 * order[q] + 1);
        order.push_back(2 * order[q] + 2);
        meta = split_meta(order[q], left);
      } else {
        meta = kMetaLeaf;
      }
      recs.push_back(vb);
      recs.push_back(meta);
    }
  }
  out.assign(tail_off + recs.size() * 4, 0);
  std::memcpy(out.data(), heads.data(), heads.size());
  if (!recs.empty()) std::memcpy(out.data() + tail_off, recs.data(), recs.size() * 4);
  dm.kind = kTableSplit;
  dm.n_trees = n_trees;
  dm.depth = depth;
  dm.tree_bytes = hb;
  dm.head_levels = H;
  dm.tail_off = tail_off;
  return MLT_OK;
}

// Half table (kTableHalf): validate like pack_ensemble, then store the
// complete heap with binary16 thresholds and leaves (round to nearest even).
int pack_ensemble_half(const mlt_node* nodes, int n_trees, int depth, int F, std::vector<unsigned char>& out,
                       DeviceModel& dm) {
  {
    std::vector<unsigned char> scratch;
    DeviceModel probe;
    const int rc = pack_ensemble(nodes, n_trees, depth, F, scratch, probe);  // validation
    if (rc != MLT_OK) return rc;
  }
  const int slots = (2 << depth) - 1;
  const HalfLayout lay = half_layout(depth);
  const size_t tb = lay.bytes;
  const int inner = (1 << depth) - 1;  // internal heap slots of the complete tree
  dm.kind = kTableHalf;
  dm.n_trees = n_trees;
  dm.depth = depth;
  dm.tree_bytes = lay.bytes;
  out.assign(tb * n_trees, 0);
  std::vector<unsigned char> reach(slots);
  std::vector<float> inherit(slots);
  std::vector<uint32_t> word(inner);
  auto h16 = [](float v) { return static_cast<uint32_t>(__half_as_ushort(__float2half_rn(v))); };
  for (int t = 0; t < n_trees; ++t) {
    const mlt_node* tr = nodes + static_cast<size_t>(t) * slots;
    unsigned char* dst = out.data() + tb * t;
    std::fill(reach.begin(), reach.end(), 0);
    reach[0] = 1;
    for (int j = 0; j < slots; ++j) {
      const mlt_node& nd = tr[j];
      const bool split = reach[j] && nd.feature >= 0;
      if (split) {
        reach[2 * j + 1] = 1;
        reach[2 * j + 2] = 1;
      }
      if (reach[j] && nd.feature == -1) {
        const uint32_t lb = h16(nd.value);
        if ((lb & 0x7C00u) == 0x7C00u)
          return fail(MLT_EINVAL, "tree %d slot %d: leaf %g does not fit binary16", t, j, nd.value);
        inherit[j] = nd.value;
      } else if (!reach[j]) {
        inherit[j] = inherit[(j - 1) / 2];  // below a leaf: copy it down
      } else {
        inherit[j] = 0.0f;
      }
      if (j < inner)
        word[j] = split ? (h16(nd.value) | (static_cast<uint32_t>(nd.feature) << kHalfFeatureShift) |
                           (nd.default_left ? kMetaDefaultLeft : 0u))
                        : 0u;  // pass-through: threshold 0 on feature 0, both sides lead to the same leaf
    }
    for (uint32_t j = 0; j < static_cast<uint32_t>(inner); ++j) {
      if (j < lay.n_inner) {
        std::memcpy(dst + 4 * j, &word[j], 4);
      } else {
        unsigned char* rec = dst + lay.off_last + 8 * (j - lay.n_inner);
        const uint32_t leaves = h16(inherit[2 * j + 1]) | (h16(inherit[2 * j + 2]) << 16);
        std::memcpy(rec, &word[j], 4);
        std::memcpy(rec + 4, &leaves, 4);
      }
    }
  }
  return MLT_OK;
}

// Upload a packed table into model slot `model_id` (lock held).
int install_model(int model_id, const std::vector<unsigned char>& packed, const DeviceModel& dm) {
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  unsigned char* d = nullptr;
  cudaError_t e = cudaMalloc(&d, packed.size());
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(MLT_ENOMEM, "cannot allocate %zu bytes for the ensemble", packed.size());
  }
  e = cudaMemcpy(d, packed.data(), packed.size(), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    cudaFree(d);
    return cuda_fail(e, "ensemble upload");
  }
  free_model(g_models[model_id]);
  Model& m = g_models[model_id];
  m.loaded = true;
  m.device = dev;
  m.F = g_F;
  m.owned = d;
  m.dm = dm;
  m.dm.table = d;
  m.dm.bytes = packed.size();
  if (dm.kind == kTableSplit) m.dm.tail = d + dm.tail_off;
  return MLT_OK;
}

}  // namespace

extern "C" {

int mlt_set_num_features(int F) {
  if (F < 1 || F > kMaxF) return fail(MLT_EINVAL, "F must lie in [1, %d], got %d", kMaxF, F);
  std::lock_guard<std::mutex> lk(g_mu);
  if (F != g_F)
    for (Model& m : g_models) free_model(m);
  g_F = F;
  return MLT_OK;
}

int mlt_load_ensemble(int model_id, const mlt_node* nodes, int n_trees, int depth) {
  if (model_id < MLT_MODEL_V || model_id > MLT_MODEL_A) return fail(MLT_EINVAL, "unknown model id %d", model_id);
  if (nodes == nullptr) return fail(MLT_EINVAL, "nodes must be non-NULL");
  if (n_trees < 1 || n_trees > 65536) return fail(MLT_EINVAL, "n_trees must lie in [1, 65536], got %d", n_trees);
  if (depth < 1 || depth > kMaxDepth) return fail(MLT_EINVAL, "depth must lie in [1, %d], got %d", kMaxDepth, depth);
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_EINVAL, "call mlt_set_num_features before loading ensembles");
  std::vector<unsigned char> packed;
  DeviceModel dm;
  // models V and P deeper than a full table: split tables (model A keeps
  // the compact table its rerank walks)
  const bool split = depth > kMaxFullDepth && model_id != MLT_MODEL_A && g_head_levels > 0;
  int rc = split ? pack_split(nodes, n_trees, depth, g_F, g_head_levels, packed, dm)
                 : pack_ensemble(nodes, n_trees, depth, g_F, packed, dm);
  if (rc != MLT_OK) return rc;
  return install_model(model_id, packed, dm);
}

int mlt_tune_decode_jit(int64_t min_n) {
  if (min_n < 0) return fail(MLT_EINVAL, "min_n must be >= 0, got %lld", static_cast<long long>(min_n));
  std::lock_guard<std::mutex> lk(g_mu);
  g_jit_min_n = min_n;
  return MLT_OK;
}

int mlt_decode_jit_available(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  return jit_available() ? 1 : 0;
}

int64_t mlt_decode_jit_calls(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  return g_jit_calls;
}

int mlt_tune_fused_small(int max_n) {
  if (max_n < 0 || max_n > kSmallMaxN) return fail(MLT_EINVAL, "max_n must lie in [0, %d], got %d", kSmallMaxN, max_n);
  std::lock_guard<std::mutex> lk(g_mu);
  g_small_max = max_n;
  return MLT_OK;
}

int mlt_tune_head_levels(int levels) {
  if (!(levels == 0 || levels == 6 || levels == 7))
    return fail(MLT_EINVAL, "levels must be 0 (compact tables), 6 or 7, got %d", levels);
  std::lock_guard<std::mutex> lk(g_mu);
  g_head_levels = levels;
  return MLT_OK;
}

int mlt_load_ensemble_f16(int model_id, const mlt_node* nodes, int n_trees, int depth) {
  if (model_id != MLT_MODEL_V && model_id != MLT_MODEL_P)
    return fail(MLT_EINVAL, "half tables are for models V and P, got model id %d", model_id);
  if (nodes == nullptr) return fail(MLT_EINVAL, "nodes must be non-NULL");
  if (n_trees < 1 || n_trees > 65536) return fail(MLT_EINVAL, "n_trees must lie in [1, 65536], got %d", n_trees);
  if (depth < 1 || depth > kMaxFullDepth)
    return fail(MLT_EINVAL, "half tables need depth in [1, %d], got %d", kMaxFullDepth, depth);
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_EINVAL, "call mlt_set_num_features before loading ensembles");
  if (g_F > static_cast<int>(kHalfFeatureMask) + 1) return fail(MLT_EINVAL, "half tables need F <= 1024");
  std::vector<unsigned char> packed;
  DeviceModel dm;
  int rc = pack_ensemble_half(nodes, n_trees, depth, g_F, packed, dm);
  if (rc != MLT_OK) return rc;
  return install_model(model_id, packed, dm);
}

int mlt_free_ensemble(int model_id) {
  if (model_id < MLT_MODEL_V || model_id > MLT_MODEL_A) return fail(MLT_EINVAL, "unknown model id %d", model_id);
  std::lock_guard<std::mutex> lk(g_mu);
  free_model(g_models[model_id]);
  return MLT_OK;
}

int mlt_validity_cut(float thr, float* tau_out) {
  if (tau_out == nullptr) return fail(MLT_EINVAL, "tau_out must be non-NULL");
  if (!(thr > 0.0f && thr < 1.0f)) return fail(MLT_EINVAL, "thr must lie in (0, 1)");
  *tau_out = validity_cut(thr);
  return MLT_OK;
}

int mlt_screen(void* stream, const float* feats, int64_t n, float thr, int k, float* out_pvalid,
               float* out_perf, int64_t* out_topk) {
  int rc = check_screen_args(n, thr, k);
  if (rc != MLT_OK) return rc;
  if ((n > 0 && (feats == nullptr || out_pvalid == nullptr || out_perf == nullptr)) || out_topk == nullptr)
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  return run_screen(static_cast<cudaStream_t>(stream), feats, nullptr, n, thr, k, out_pvalid, out_perf, out_topk);
}

int mlt_screen_noalloc(void* stream, const float* feats, int64_t n, float thr, int k, float* out_pvalid,
                       float* out_perf, int64_t* out_topk) {
  int rc = check_screen_args(n, thr, k);
  if (rc != MLT_OK) return rc;
  if (n > mlt_noalloc::kMaxN)
    return fail(MLT_EINVAL, "n=%lld exceeds the %lld candidates the static scratch holds", static_cast<long long>(n),
                mlt_noalloc::kMaxN);
  if ((n > 0 && (feats == nullptr || out_pvalid == nullptr || out_perf == nullptr)) || out_topk == nullptr)
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  int dev = 0;
  rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  Scratch s;
  rc = noalloc_scratch(dev, &s);
  if (rc != MLT_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents; the selection state is
  // cleared at the start of the sequence, the error word only when
  // mlt_sync_status reads it (so a fault of this call stays visible)
  return run_screen_with(st, feats, nullptr, n, thr, k, out_pvalid, out_perf, out_topk, s, false);
}

int mlt_merge_topk(void* stream, const float* scores, const int64_t* indices, int64_t m, int k,
                   int64_t* out_topk) {
  if (m < 0 || m > kMaxMergePairs) return fail(MLT_EINVAL, "m must lie in [0, %lld], got %lld", kMaxMergePairs,
                                               static_cast<long long>(m));
  if (k < 1 || k > kMaxK) return fail(MLT_EINVAL, "k must lie in [1, %d], got %d", kMaxK, k);
  if ((m > 0 && (scores == nullptr || indices == nullptr)) || out_topk == nullptr)
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  MLT_CUDA(launch_merge_topk(scores, indices, m, k, out_topk, static_cast<cudaStream_t>(stream)), "merge launch");
  std::lock_guard<std::mutex> lk(g_mu);
  g_launches += m > 0 ? 1 : 0;
  return MLT_OK;
}

int mlt_screen_until(void* stream, const float* feats, int64_t n_total, int64_t batch, int64_t target, float thr,
                     int k, float* out_pvalid, float* out_perf, int64_t* out_topk, int64_t* out_stats) {
  int rc = check_stream_args(n_total, batch, target, thr, k);
  if (rc != MLT_OK) return rc;
  if ((n_total > 0 && feats == nullptr) || out_topk == nullptr) return fail(MLT_EINVAL, "feats and out_topk must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  return run_stream(static_cast<cudaStream_t>(stream), feats, nullptr, n_total, batch, target, thr, k, out_pvalid,
                    out_perf, out_topk, out_stats);
}

int mlt_screen_until_decoded(void* stream, const int32_t* radices, const float* option_values, int n_knobs,
                             const mlt_feat_op* program, int64_t first_index, int64_t n_total, int64_t batch,
                             int64_t target, float thr, int k, float* out_pvalid, float* out_perf,
                             int64_t* out_topk, int64_t* out_stats) {
  int rc = check_stream_args(n_total, batch, target, thr, k);
  if (rc != MLT_OK) return rc;
  if (out_topk == nullptr) return fail(MLT_EINVAL, "out_topk must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  DecodeParams d;
  rc = build_decoder(radices, option_values, n_knobs, program, g_F, first_index, n_total, &d);
  if (rc != MLT_OK) return rc;
  return run_stream(static_cast<cudaStream_t>(stream), nullptr, &d, n_total, batch, target, thr, k, out_pvalid,
                    out_perf, out_topk, out_stats);
}

int mlt_sa_step(void* stream, const int32_t* radices, const float* option_values, int n_knobs,
                const mlt_feat_op* program, const int64_t* parent, const float* parent_score,
                const uint32_t* knob_draw, const uint32_t* digit_draw, const float* log_u, int64_t m,
                float temperature, float thr, int64_t* out_next, float* out_next_score, int32_t* out_accepted) {
  if (m < 0 || m > 0x7FFFFFFFLL) return fail(MLT_EINVAL, "m must lie in [0, 2^31-1]");
  if (!(thr > 0.0f && thr < 1.0f)) return fail(MLT_EINVAL, "thr must lie in (0, 1)");
  if (!(temperature > 0.0f) || !std::isfinite(temperature)) return fail(MLT_EINVAL, "temperature must be positive");
  if (m > 0 && (parent == nullptr || parent_score == nullptr || knob_draw == nullptr || digit_draw == nullptr ||
                log_u == nullptr || out_next == nullptr || out_next_score == nullptr || out_accepted == nullptr))
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  DecodeParams d;
  int rc = build_decoder(radices, option_values, n_knobs, program, g_F, 0, 0, &d);
  if (rc != MLT_OK) return rc;
  long double space_ld = 1.0L;
  for (int j = 0; j < n_knobs; ++j) space_ld *= radices[j];
  const long long space = space_ld > 9.0e18L ? static_cast<long long>(9.0e18L) : static_cast<long long>(space_ld);
  if (m == 0) return MLT_OK;
  rc = ensure_scratch(m);
  if (rc != MLT_OK) return rc;
  ScratchOwner& S = g_scr;
  if (m > S.sa_cap) {
    cudaDeviceSynchronize();
    cudaFree(S.sa_prop);
    cudaFree(S.sa_pvalid);
    cudaFree(S.sa_perf);
    cudaFree(S.sa_topk);
    S.sa_prop = nullptr;
    S.sa_pvalid = S.sa_perf = nullptr;
    S.sa_topk = nullptr;
    S.sa_cap = -1;
    if (cudaMalloc(&S.sa_prop, sizeof(long long) * m) != cudaSuccess ||
        cudaMalloc(&S.sa_pvalid, sizeof(float) * m) != cudaSuccess ||
        cudaMalloc(&S.sa_perf, sizeof(float) * m) != cudaSuccess ||
        cudaMalloc(&S.sa_topk, sizeof(int64_t)) != cudaSuccess) {
      cudaGetLastError();
      return fail(MLT_ENOMEM, "cannot allocate proposal buffers");
    }
    S.sa_cap = m;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  MLT_CUDA(launch_sa_propose(d, space, parent, knob_draw, digit_draw, m, S.sa_prop, S.err, st), "propose launch");
  d.index_list = S.sa_prop;
  rc = run_screen_with(st, nullptr, &d, m, thr, 1, S.sa_pvalid, S.sa_perf, S.sa_topk, g_scr.s, true);
  if (rc != MLT_OK) return rc;
  MLT_CUDA(launch_sa_accept(space, parent, parent_score, S.sa_prop, S.sa_perf, log_u, m, temperature, out_next,
                            out_next_score, out_accepted, st),
           "accept launch");
  g_launches += 2;
  return MLT_OK;
}

int mlt_rerank(void* stream, const float* feats, int64_t n, const int64_t* cand, int m, int n_final,
               float* out_score, int64_t* out_final) {
  if (n < 0 || n > 0x7FFFFFFFLL) return fail(MLT_EINVAL, "n must lie in [0, 2^31-1]");
  if (m < 0 || m > kMaxK) return fail(MLT_EINVAL, "m must lie in [0, %d], got %d", kMaxK, m);
  if (n_final < 1 || n_final > kMaxK) return fail(MLT_EINVAL, "n_final must lie in [1, %d], got %d", kMaxK, n_final);
  if ((m > 0 && (cand == nullptr || out_score == nullptr || (n > 0 && feats == nullptr))) || out_final == nullptr)
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  const Model& A = g_models[MLT_MODEL_A];
  if (!A.loaded) return fail(MLT_ENOMODEL, "model A is not loaded");
  if (A.F != g_F) return fail(MLT_ENOMODEL, "model A was loaded for F=%d, current F=%d", A.F, g_F);
  if (A.device != dev) return fail(MLT_EINVAL, "model A lives on device %d, current device is %d", A.device, dev);
  rc = ensure_scratch(0);
  if (rc != MLT_OK) return rc;
  MLT_CUDA(launch_rerank(A.dm, feats, g_F, n, cand, m, n_final, out_score, out_final, g_scr.rerank_keys, g_scr.err,
                         static_cast<cudaStream_t>(stream)),
           "rerank launch");
  g_launches += (m > 0 ? 1 : 0) + 1;
  return MLT_OK;
}

int mlt_screen_decoded(void* stream, const int32_t* radices, const float* option_values, int n_knobs,
                       const mlt_feat_op* program, int64_t first_index, int64_t n, float thr, int k,
                       float* out_pvalid, float* out_perf, int64_t* out_topk) {
  int rc = check_screen_args(n, thr, k);
  if (rc != MLT_OK) return rc;
  if ((n > 0 && (out_pvalid == nullptr || out_perf == nullptr)) || out_topk == nullptr)
    return fail(MLT_EINVAL, "device buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  DecodeParams d;
  rc = build_decoder(radices, option_values, n_knobs, program, g_F, first_index, n, &d);
  if (rc != MLT_OK) return rc;
  return run_screen(static_cast<cudaStream_t>(stream), nullptr, &d, n, thr, k, out_pvalid, out_perf, out_topk);
}

int mlt_screen_host(void* stream, const float* feats_host, int64_t n, float thr, int k, float* pvalid_host,
                    float* perf_host, int64_t* topk_host) {
  int rc = check_screen_args(n, thr, k);
  if (rc != MLT_OK) return rc;
  if ((n > 0 && (feats_host == nullptr || pvalid_host == nullptr || perf_host == nullptr)) || topk_host == nullptr)
    return fail(MLT_EINVAL, "host buffers must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ScratchOwner& S = g_scr;
  if (n > S.host_cap_n || g_F != S.host_cap_F || S.h_topk == nullptr) {
    cudaDeviceSynchronize();
    cudaFree(S.h_feats);
    cudaFree(S.h_pvalid);
    cudaFree(S.h_perf);
    cudaFree(S.h_topk);
    S.h_feats = nullptr;
    S.h_pvalid = S.h_perf = nullptr;
    S.h_topk = nullptr;
    S.host_cap_n = -1;
    const long long cap = n < 1024 ? 1024 : n;
    if (cudaMalloc(&S.h_feats, sizeof(float) * cap * g_F) != cudaSuccess ||
        cudaMalloc(&S.h_pvalid, sizeof(float) * cap) != cudaSuccess ||
        cudaMalloc(&S.h_perf, sizeof(float) * cap) != cudaSuccess ||
        cudaMalloc(&S.h_topk, sizeof(int64_t) * kMaxK) != cudaSuccess) {
      cudaGetLastError();
      return fail(MLT_ENOMEM, "cannot allocate device staging for host buffers");
    }
    S.host_cap_n = cap;
    S.host_cap_F = g_F;
  }
  if (n > 0)
    MLT_CUDA(cudaMemcpyAsync(S.h_feats, feats_host, sizeof(float) * n * g_F, cudaMemcpyHostToDevice, st),
             "feature upload");
  rc = run_screen(st, S.h_feats, nullptr, n, thr, k, S.h_pvalid, S.h_perf, S.h_topk);
  if (rc != MLT_OK) return rc;
  if (n > 0) {
    MLT_CUDA(cudaMemcpyAsync(pvalid_host, S.h_pvalid, sizeof(float) * n, cudaMemcpyDeviceToHost, st), "pvalid download");
    MLT_CUDA(cudaMemcpyAsync(perf_host, S.h_perf, sizeof(float) * n, cudaMemcpyDeviceToHost, st), "perf download");
  }
  MLT_CUDA(cudaMemcpyAsync(topk_host, S.h_topk, sizeof(int64_t) * k, cudaMemcpyDeviceToHost, st), "top-k download");
  MLT_CUDA(cudaStreamSynchronize(st), "stream synchronize");
  return MLT_OK;
}

int mlt_screen_host_batches(void* stream, int64_t n_batches, const float* const* feats_host, int64_t n, float thr,
                            int k, float* const* pvalid_host, float* const* perf_host, int64_t* const* topk_host) {
  int rc = check_screen_args(n, thr, k);
  if (rc != MLT_OK) return rc;
  if (n_batches < 0) return fail(MLT_EINVAL, "n_batches must be >= 0");
  if (n_batches == 0) return MLT_OK;
  if (feats_host == nullptr || topk_host == nullptr) return fail(MLT_EINVAL, "feats_host and topk_host must be non-NULL");
  for (int64_t b = 0; b < n_batches; ++b)
    if ((n > 0 && feats_host[b] == nullptr) || topk_host[b] == nullptr)
      return fail(MLT_EINVAL, "batch %lld: host buffers must be non-NULL", static_cast<long long>(b));
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  cudaStream_t sc = static_cast<cudaStream_t>(stream);
  ScratchOwner& S = g_scr;
  if (S.hb_copy == nullptr) {
    MLT_CUDA(cudaStreamCreateWithFlags(&S.hb_copy, cudaStreamNonBlocking), "copy stream");
    for (int i = 0; i < 2; ++i) {
      MLT_CUDA(cudaEventCreateWithFlags(&S.hb_in[i], cudaEventDisableTiming), "cudaEventCreate");
      MLT_CUDA(cudaEventCreateWithFlags(&S.hb_out[i], cudaEventDisableTiming), "cudaEventCreate");
      MLT_CUDA(cudaEventCreateWithFlags(&S.hb_down[i], cudaEventDisableTiming), "cudaEventCreate");
    }
  }
  if (n > S.hb_cap_n || g_F != S.hb_cap_F) {
    cudaDeviceSynchronize();
    for (int i = 0; i < 2; ++i) {
      cudaFree(S.hb_feats[i]);
      cudaFree(S.hb_pvalid[i]);
      cudaFree(S.hb_perf[i]);
      cudaFree(S.hb_topk[i]);
      S.hb_feats[i] = nullptr;
      S.hb_pvalid[i] = S.hb_perf[i] = nullptr;
      S.hb_topk[i] = nullptr;
    }
    S.hb_cap_n = -1;
    const long long cap = n < 1024 ? 1024 : n;
    for (int i = 0; i < 2; ++i) {
      if (cudaMalloc(&S.hb_feats[i], sizeof(float) * cap * g_F) != cudaSuccess ||
          cudaMalloc(&S.hb_pvalid[i], sizeof(float) * cap) != cudaSuccess ||
          cudaMalloc(&S.hb_perf[i], sizeof(float) * cap) != cudaSuccess ||
          cudaMalloc(&S.hb_topk[i], sizeof(int64_t) * kMaxK) != cudaSuccess) {
        cudaGetLastError();
        return fail(MLT_ENOMEM, "cannot allocate device staging for host batches");
      }
    }
    S.hb_cap_n = cap;
    S.hb_cap_F = g_F;
  }
  rc = ensure_scratch(n);  // before the pipeline: growing it synchronises the device
  if (rc != MLT_OK) return rc;
  cudaStream_t sh = S.hb_copy;
  const size_t in_bytes = sizeof(float) * static_cast<size_t>(n) * g_F;
  auto upload = [&](int64_t b) -> int {
    const int i = static_cast<int>(b & 1);
    if (n > 0)
      MLT_CUDA(cudaMemcpyAsync(S.hb_feats[i], feats_host[b], in_bytes, cudaMemcpyHostToDevice, sh), "feature upload");
    MLT_CUDA(cudaEventRecord(S.hb_in[i], sh), "cudaEventRecord");
    return MLT_OK;
  };
  auto download = [&](int64_t b) -> int {
    const int i = static_cast<int>(b & 1);
    MLT_CUDA(cudaStreamWaitEvent(sh, S.hb_out[i], 0), "cudaStreamWaitEvent");
    if (n > 0 && pvalid_host != nullptr && pvalid_host[b] != nullptr)
      MLT_CUDA(cudaMemcpyAsync(pvalid_host[b], S.hb_pvalid[i], sizeof(float) * n, cudaMemcpyDeviceToHost, sh),
               "pvalid download");
    if (n > 0 && perf_host != nullptr && perf_host[b] != nullptr)
      MLT_CUDA(cudaMemcpyAsync(perf_host[b], S.hb_perf[i], sizeof(float) * n, cudaMemcpyDeviceToHost, sh),
               "perf download");
    MLT_CUDA(cudaMemcpyAsync(topk_host[b], S.hb_topk[i], sizeof(int64_t) * k, cudaMemcpyDeviceToHost, sh),
             "top-k download");
    MLT_CUDA(cudaEventRecord(S.hb_down[i], sh), "cudaEventRecord");
    return MLT_OK;
  };
  // the copy stream starts after the caller's earlier work on `stream`
  MLT_CUDA(cudaEventRecord(S.hb_out[1], sc), "cudaEventRecord");
  MLT_CUDA(cudaStreamWaitEvent(sh, S.hb_out[1], 0), "cudaStreamWaitEvent");
  rc = upload(0);
  if (rc != MLT_OK) return rc;
  // batch b screens on `stream` while the copy stream brings back batch
  // b-1's results and uploads batch b+1 (two staging sets in turn)
  for (int64_t b = 0; b < n_batches; ++b) {
    const int i = static_cast<int>(b & 1);
    MLT_CUDA(cudaStreamWaitEvent(sc, S.hb_in[i], 0), "cudaStreamWaitEvent");
    if (b >= 2) MLT_CUDA(cudaStreamWaitEvent(sc, S.hb_down[i], 0), "cudaStreamWaitEvent");
    rc = run_screen_with(sc, S.hb_feats[i], nullptr, n, thr, k, S.hb_pvalid[i], S.hb_perf[i], S.hb_topk[i], S.s, true);
    if (rc != MLT_OK) return rc;
    MLT_CUDA(cudaEventRecord(S.hb_out[i], sc), "cudaEventRecord");
    if (b >= 1) {
      rc = download(b - 1);  // waits for batch b-1, whose staging batch b+1 reuses
      if (rc != MLT_OK) return rc;
    }
    if (b + 1 < n_batches) {
      rc = upload(b + 1);
      if (rc != MLT_OK) return rc;
    }
  }
  rc = download(n_batches - 1);
  if (rc != MLT_OK) return rc;
  MLT_CUDA(cudaStreamSynchronize(sh), "copy stream synchronize");
  MLT_CUDA(cudaStreamSynchronize(sc), "stream synchronize");
  return MLT_OK;
}

int mlt_decode_knobs(void* stream, const int32_t* radices, const float* option_values, int n_knobs,
                     const mlt_feat_op* program, int F, int64_t first_index, int64_t n, uint8_t* out_knobs,
                     float* out_feats) {
  if (n < 0 || n > 0x7FFFFFFFLL) return fail(MLT_EINVAL, "n must lie in [0, 2^31-1]");
  DecodeParams d;
  int rc = build_decoder(radices, option_values, n_knobs, program, F, first_index, n, &d);
  if (rc != MLT_OK) return rc;
  if (n == 0) return MLT_OK;
  MLT_CUDA(launch_decode_rows(d, n, out_knobs, out_feats, static_cast<cudaStream_t>(stream)), "decode launch");
  std::lock_guard<std::mutex> lk(g_mu);
  g_launches += 1;
  return MLT_OK;
}

int mlt_sync_status(void* stream) {
  MLT_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream synchronize");
  std::lock_guard<std::mutex> lk(g_mu);
  // the allocating entry points' error word, and the static scratch's of
  // mlt_screen_noalloc on the current device (read and cleared without any
  // allocation)
  unsigned int* words[2] = {g_scr.err, nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < mlt_noalloc::kMaxDevices &&
      g_noalloc_base[dev] != nullptr)
    words[1] = reinterpret_cast<unsigned int*>(g_noalloc_base[dev] + mlt_noalloc::kErr);
  unsigned int word = 0;
  for (unsigned int* w : words) {
    if (w == nullptr) continue;
    unsigned int v = 0;
    MLT_CUDA(cudaMemcpy(&v, w, sizeof(v), cudaMemcpyDeviceToHost), "error word read");
    if (v != 0) MLT_CUDA(cudaMemset(w, 0, sizeof(v)), "error word reset");
    word |= v;
  }
  if (word == 0) return MLT_OK;
  if (word & kErrWaitTimeout) return fail(MLT_ETIMEOUT, "a device-side wait gave up (error word 0x%x)", word);
  if (word & kErrBadIndex) return fail(MLT_EINVAL, "a rerank candidate index was outside [0, n) (error word 0x%x)", word);
  return fail(MLT_ECUDA, "device-side bookkeeping error (error word 0x%x)", word);
}

int mlt_selftest_wait_timeout(void* stream, int64_t limit_ns) {
  if (limit_ns < 1000000LL || limit_ns > static_cast<int64_t>(kWaitLimitNs))
    return fail(MLT_EINVAL, "limit_ns must lie in [1e6, %llu]", kWaitLimitNs);
  std::lock_guard<std::mutex> lk(g_mu);
  const int rc = ensure_scratch(0);  // the device error word
  if (rc != MLT_OK) return rc;
  MLT_CUDA(launch_wait_selftest(g_scr.err, static_cast<unsigned long long>(limit_ns),
                                static_cast<cudaStream_t>(stream)),
           "self-test launch");
  g_launches += 1;
  return MLT_OK;
}

int mlt_selftest_walk_timeout(int cta, int64_t limit_ns) {
  if (cta < 0) return fail(MLT_EINVAL, "cta must be >= 0");
  if (limit_ns < 1000000LL || limit_ns > static_cast<int64_t>(kWaitLimitNs))
    return fail(MLT_EINVAL, "limit_ns must lie in [1e6, %llu]", kWaitLimitNs);
  std::lock_guard<std::mutex> lk(g_mu);
  g_stall_cta = cta;
  g_stall_ns = static_cast<unsigned long long>(limit_ns);
  return MLT_OK;
}

int mlt_selftest_poison_state(int static_scratch, uint32_t value) {
  std::lock_guard<std::mutex> lk(g_mu);
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  Scratch s;
  if (static_scratch) {
    rc = noalloc_scratch(dev, &s);
  } else {
    rc = ensure_scratch(0);
    s = g_scr.s;
  }
  if (rc != MLT_OK) return rc;
  const unsigned int words[4] = {value, value, value, value};  // survivors, n_cand, ticket, v_ticket
  MLT_CUDA(cudaMemcpy(s.state, words, sizeof(words), cudaMemcpyHostToDevice), "state write");
  return MLT_OK;
}

int mlt_last_survivor_count(void* stream, int64_t* count_out) {
  if (count_out == nullptr) return fail(MLT_EINVAL, "count_out must be non-NULL");
  MLT_CUDA(cudaStreamSynchronize(static_cast<cudaStream_t>(stream)), "stream synchronize");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_scr.state == nullptr) {
    *count_out = 0;
    return MLT_OK;
  }
  unsigned int s = 0;
  MLT_CUDA(cudaMemcpy(&s, &g_scr.state->survivors, sizeof(s), cudaMemcpyDeviceToHost), "survivor count read");
  *count_out = s;
  return MLT_OK;
}

int mlt_profile_phases(int enable) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_profile = enable != 0;
  g_events_used = 0;
  return MLT_OK;
}

int mlt_phase_times(float* out_ms, int n_phases, int64_t* n_calls_out) {
  if (out_ms == nullptr || n_calls_out == nullptr || n_phases < 0)
    return fail(MLT_EINVAL, "out_ms and n_calls_out must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  double sum[kPhases] = {0, 0, 0, 0};
  const size_t calls = g_events_used / (kPhases + 1);
  for (size_t c = 0; c < calls; ++c) {
    cudaEvent_t* ev = &g_events[c * (kPhases + 1)];
    MLT_CUDA(cudaEventSynchronize(ev[kPhases]), "cudaEventSynchronize");
    for (int p = 0; p < kPhases; ++p) {
      float ms = 0.0f;
      MLT_CUDA(cudaEventElapsedTime(&ms, ev[p], ev[p + 1]), "cudaEventElapsedTime");
      sum[p] += ms;
    }
  }
  for (int p = 0; p < n_phases && p < kPhases; ++p) out_ms[p] = static_cast<float>(sum[p]);
  *n_calls_out = static_cast<int64_t>(calls);
  g_events_used = 0;
  return MLT_OK;
}

int mlt_walk_peak(void* stream, int model_id, const float* feats, int64_t n, int rounds, float* out_sums,
                  int64_t* visits_out) {
  if (model_id != MLT_MODEL_V && model_id != MLT_MODEL_P) return fail(MLT_EINVAL, "model_id must be V or P");
  if (n < 1 || n > 0x7FFFFFFFLL) return fail(MLT_EINVAL, "n must lie in [1, 2^31-1]");
  if (rounds < 1 || rounds > 1000000) return fail(MLT_EINVAL, "rounds must lie in [1, 1e6]");
  if (feats == nullptr || out_sums == nullptr || visits_out == nullptr)
    return fail(MLT_EINVAL, "feats, out_sums and visits_out must be non-NULL");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_F <= 0) return fail(MLT_ENOMODEL, "no feature count set");
  const Model& m = g_models[model_id];
  if (!m.loaded || m.F != g_F) return fail(MLT_ENOMODEL, "model %d is not loaded for F=%d", model_id, g_F);
  if (m.dm.kind != kTableFull) return fail(MLT_EINVAL, "the walk-rate ceiling needs a full fp32 table (depth <= %d)", kMaxFullDepth);
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  if (m.device != dev) return fail(MLT_EINVAL, "model %d lives on device %d, current device is %d", model_id, m.device, dev);
  const DeviceModel& dm = m.dm;
  const ScreenShape s = plan_for(dm, g_F, n, g_shape[model_id], true);
  if (s.threads == 0) return fail(MLT_EINVAL, "F=%d leaves no room for a shared-memory tile", g_F);
  // one thread per candidate (a tree-group shape becomes one wider group)
  const int tc = std::min(kFullMaxTile, s.threads * s.lanes);
  const size_t feat_bytes = walk_peak_tree_offset(g_F, tc);
  int resident = std::min(dm.n_trees, s.chunk_trees * s.nbuf);
  while (resident > 1 && feat_bytes + static_cast<size_t>(resident) * dm.tree_bytes + 1024 > static_cast<size_t>(smem_optin()))
    --resident;
  const size_t smem = feat_bytes + static_cast<size_t>(resident) * dm.tree_bytes;
  if (smem + 1024 > static_cast<size_t>(smem_optin())) return fail(MLT_EINVAL, "F=%d leaves no room for a tree", g_F);
  WalkPeakKernelPtr k = walk_peak_kernel(dm.depth, s.group);
  if (k == nullptr) return fail(MLT_EINVAL, "no walk-rate kernel for depth %d, group %d", dm.depth, s.group);
  rc = ensure_scratch(0);  // the device error word
  if (rc != MLT_OK) return rc;
  TraverseArgs a{};
  a.feats = feats;
  a.F = g_F;
  a.n = n;
  a.vec4 = ((reinterpret_cast<uintptr_t>(feats) & 15u) == 0 && (g_F & 3) == 0) ? 1 : 0;
  a.table = dm.table;
  a.n_trees = dm.n_trees;
  a.tree_bytes = dm.tree_bytes;
  a.err = g_scr.err;
  MLT_CUDA(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)),
           "walk-rate kernel attribute");
  const long long tiles = (n + tc - 1) / tc;
  k<<<dim3(static_cast<unsigned>(tiles)), dim3(tc), smem, static_cast<cudaStream_t>(stream)>>>(a, resident, rounds,
                                                                                             out_sums);
  MLT_CUDA(cudaGetLastError(), "walk-rate kernel launch");
  g_launches += 1;
  *visits_out = static_cast<int64_t>(n) * resident * dm.depth * rounds;
  return MLT_OK;
}

int mlt_walk_shape(int model_id, int64_t n, int p_pass, int32_t* out) {
  if (model_id != MLT_MODEL_V && model_id != MLT_MODEL_P)
    return fail(MLT_EINVAL, "model id must be V (0) or P (1), got %d", model_id);
  if (out == nullptr) return fail(MLT_EINVAL, "out must be non-NULL");
  if (n < 1) return fail(MLT_EINVAL, "n must be >= 1, got %lld", static_cast<long long>(n));
  std::lock_guard<std::mutex> lk(g_mu);
  int dev = 0;
  int rc = current_device(&dev);
  if (rc != MLT_OK) return rc;
  const Model& m = g_models[model_id];
  if (!m.loaded) return fail(MLT_ENOMODEL, "model %d is not loaded", model_id);
  if (m.device != dev) return fail(MLT_EINVAL, "model %d lives on device %d, current device is %d", model_id, m.device, dev);
  // the P pass is planned for about half the batch, as the screening does
  const ScreenShape sh = plan_for(m.dm, g_F, p_pass ? (n + 1) / 2 : n, g_shape[model_id], !p_pass);
  if (sh.threads == 0) return fail(MLT_EINVAL, "F=%d leaves no room for a shared-memory tile", g_F);
  out[0] = sh.threads;
  out[1] = sh.lanes;
  out[2] = sh.group;
  out[3] = sh.chunk_trees;
  out[4] = sh.nbuf;
  out[5] = sh.resident;
  out[6] = m.dm.kind;
  return MLT_OK;
}

int mlt_tune_walk(int model_id, int candidates, int splits, int group, int chunk_trees, int nbuf) {
  if (model_id < MLT_MODEL_V || model_id > MLT_MODEL_A) return fail(MLT_EINVAL, "unknown model id %d", model_id);
  if (candidates < 0 || candidates > kFullMaxTile || candidates % 32 != 0)
    return fail(MLT_EINVAL, "candidates must be 0 or a multiple of 32 up to %d", kFullMaxTile);
  if (!(splits == 0 || splits == 1 || splits == 2 || splits == 4 || splits == 8))
    return fail(MLT_EINVAL, "splits must be 0, 1, 2, 4 or 8");
  if (!(group == 0 || group == 2 || group == 4 || group == 8)) return fail(MLT_EINVAL, "group must be 0, 2, 4 or 8");
  if (!(chunk_trees == 0 || chunk_trees == 1 || chunk_trees == 2 || chunk_trees == 4 || chunk_trees == 8 ||
        chunk_trees == 16 || chunk_trees == 32))
    return fail(MLT_EINVAL, "chunk_trees must be 0, 1, 2, 4, 8, 16 or 32");
  if (!(nbuf == 0 || nbuf == 2 || nbuf == 3)) return fail(MLT_EINVAL, "nbuf must be 0, 2 or 3");
  if (candidates && splits && candidates * splits > 1024)
    return fail(MLT_EINVAL, "candidates x splits must be at most 1024");
  std::lock_guard<std::mutex> lk(g_mu);
  ShapeOverride& o = g_shape[model_id];
  o.threads = candidates;
  o.lanes = splits;
  o.group = group;
  o.chunk_trees = chunk_trees;
  o.nbuf = nbuf;
  return MLT_OK;
}

int64_t mlt_kernel_launches(void) {
  std::lock_guard<std::mutex> lk(g_mu);
  return g_launches;
}

const char* mlt_last_error(void) { return t_err.c_str(); }

}  // extern "C"
