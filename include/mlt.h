/*
 * mlt.h -- C ABI of libmlt, GB300 (sm_103a) batched candidate screening for
 * ML^2Tuner-style autotuning (arXiv 2411.10764).
 *
 * The paper's configuration explorer scores candidate code configurations
 * with a validity model V and a performance model P, drops the candidates V
 * predicts invalid, and keeps the (alpha+1)N candidates that P ranks best
 * (Sec. 2, "Configuration Explorer", "ML Model V", "ML Model P", "Hidden
 * Feature Extractor & ML Model A").  All models are XGBoost tree ensembles
 * (Sec. 3 "Experimental Setup"; Appendix A.3, Table 3).  This library runs
 * that inner step over a whole batch of candidates on one GPU.
 *
 * Conventions for every call:
 *   - Every function returns an mlt_status (0 = MLT_OK, negative = error)
 *     and never aborts or traps.  mlt_last_error() gives a message for the
 *     last failing call on the calling thread.
 *   - "device" pointers are CUDA device memory owned by the caller (for
 *     example torch tensors); "host" pointers are ordinary host memory.
 *     The library keeps no reference to a caller buffer after the call (or,
 *     for asynchronous calls, after the queued GPU work has finished).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Asynchronous calls only enqueue work on it; errors detected
 *     by the GPU (a bounded wait that gave up) are reported by the next
 *     mlt_sync_status() on that stream.
 *   - Library state (loaded ensembles, feature count, scratch buffers) is
 *     process-wide and guarded by a lock; scratch buffers are shared, so
 *     screening calls must be ordered on one stream (or the caller must
 *     synchronize between streams).
 *   - Candidate counts are limited to n < 2^31; top-k to 1 <= k <= 16384.
 */
#ifndef MLT_H
#define MLT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MLT_OK = 0,
    MLT_EINVAL = -1,   /* bad argument or malformed ensemble / program     */
    MLT_ENOMODEL = -2, /* screening asked for a model that is not loaded   */
    MLT_ECUDA = -3,    /* a CUDA runtime call failed (message has details) */
    MLT_ENOMEM = -4,   /* device or host allocation failed                 */
    MLT_ETIMEOUT = -5  /* a bounded device-side wait gave up               */
} mlt_status;

/* Model slots (Sec. 2): V = validity classifier, P = performance regressor,
 * A = the hidden-feature performance model used to rerank the kept set. */
enum { MLT_MODEL_V = 0, MLT_MODEL_P = 1, MLT_MODEL_A = 2 };

/* One tree slot in implicit heap order (12 bytes).  A tree of depth d has
 * 2^(d+1)-1 slots; the children of slot j are 2j+1 (left) and 2j+2 (right).
 *   feature >= 0 : split; x[feature] < value goes left, x >= value goes
 *                  right, a NaN (missing) x goes left iff default_left != 0;
 *   feature == -1: leaf with output `value`;
 *   feature == -2: unused slot (below a leaf, or past the tree's depth).
 * This is XGBoost's gbtree routing rule (Sec. 3 setup, Table 3); the paper
 * does not spell out the comparison, the strict `<` is this library's
 * reading. */
typedef struct {
    int32_t feature;
    float value;
    uint8_t default_left;
    uint8_t pad[3];
} mlt_node;

/* One instruction of a feature program (16 bytes); see mlt_decode_knobs. */
typedef struct {
    int32_t op;
    int32_t a;
    int32_t b;
    float c;
} mlt_feat_op;

/* Feature-program opcodes.  Operands a, b: -1 = the constant c; 0..K-1 =
 * knob j's option value; K+f = feature f of the same candidate, f below the
 * feature being computed.  Every operation is one IEEE-754 binary32
 * operation rounded to nearest (no fused multiply-add). */
enum {
    MLT_OP_COPY = 0,    /* A                                               */
    MLT_OP_ILOG2 = 1,   /* floor(log2 A) for a positive normal A, else 0    */
    MLT_OP_ADD = 2,     /* A + B                                           */
    MLT_OP_SUB = 3,     /* A - B                                           */
    MLT_OP_MUL = 4,     /* A * B                                           */
    MLT_OP_DIV = 5,     /* A / B                                           */
    MLT_OP_CEILDIV = 6, /* ceil(A / B)                                     */
    MLT_OP_REM = 7,     /* A - B * floor(A / B), three rounded operations  */
    MLT_OP_MIN = 8,     /* (B < A) ? B : A                                 */
    MLT_OP_MAX = 9,     /* (B > A) ? B : A                                 */
    MLT_OP_GT = 10,     /* (A > B) ? 1 : 0                                 */
    MLT_OP_EQ = 11      /* (A == B) ? 1 : 0                                */
};

/* Number of features F per candidate (1 <= F <= 1024).  Must be set before
 * loading ensembles; changing it unloads every ensemble.  Synchronous. */
int mlt_set_num_features(int F);

/* Copy, validate and pack one ensemble into library-owned device memory
 * (Sec. 2: model V, P or A; Table 3: XGBoost gbtree).
 *   model_id : MLT_MODEL_V, MLT_MODEL_P or MLT_MODEL_A
 *   nodes    : host array of n_trees * (2^(depth+1)-1) heap-order slots;
 *              the caller keeps ownership (it is only read during the call)
 *   n_trees  : 1 .. 65536;  depth : 1 .. 14
 * Validation (MLT_EINVAL): slot 0 is a split or a leaf; every split's two
 * children are splits or leaves; slots at `depth` that are reachable are
 * leaves; split features lie in [0, F); thresholds and leaves are finite;
 * the sum over trees of the largest |leaf| is below 1e37 (no fp32 overflow
 * in the leaf sum).  Replaces a previously loaded model in the same slot.
 * Synchronous (waits for queued work before freeing an old table). */
int mlt_load_ensemble(int model_id, const mlt_node *nodes, int n_trees, int depth);

/* Half tables: like mlt_load_ensemble, but the ensemble is stored with its
 * thresholds and leaves rounded to IEEE binary16 (round to nearest even),
 * and every screening pass over this model rounds the candidate's features
 * to binary16 too.  Halves the table and the staged features, and changes
 * results: the call screens exactly as the rounded model scores the rounded
 * rows (comparisons in binary16, leaves summed in fp32 in tree order), so
 * decisions and scores may differ from the fp32 model near split
 * thresholds and by the rounding of the leaves.  For models V and P of
 * depth 1 .. 10 with F <= 1024; a leaf whose magnitude rounds past 65504 is
 * MLT_EINVAL (a threshold that does is kept as an infinity).  Screening
 * calls that build features from candidate indices (mlt_screen_decoded,
 * mlt_screen_until_decoded, mlt_sa_step) return MLT_EINVAL while a half
 * table is loaded.  Synchronous. */
int mlt_load_ensemble_f16(int model_id, const mlt_node *nodes, int n_trees, int depth);

/* Free a loaded ensemble (no-op if the slot is empty).  Synchronous. */
int mlt_free_ensemble(int model_id);

/* The validity cut in margin space: *tau_out = the smallest float m with
 * sigmoid(m) >= thr, 0 < thr < 1 (thr = 0.5 gives 0, the sign rule of the
 * paper's binary:hinge model V, Table 3).  A candidate is valid iff its V
 * margin >= tau.  Host-only. */
int mlt_validity_cut(float thr, float *tau_out);

/* Screen a batch of candidates (the explorer's inner step, Sec. 2):
 *   margin_V(i) = sum over V's trees of the leaf row i reaches, fp32, in
 *                 tree order from 0.0f;  valid(i) = margin_V(i) >= tau(thr)
 *   out_pvalid[i] = sigmoid(margin_V(i))                       (fp32)
 *   out_perf[i]   = margin_P(i) if valid(i), else -infinity     (fp32)
 *   out_topk[r]   = index of the r-th best valid candidate by
 *                   (margin_P descending, index ascending), r < k;
 *                   -1 where fewer than k candidates are valid.
 * Arguments:
 *   feats      device, row-major [n][F] fp32 (NaN = missing value)
 *   n          0 .. 2^31-1 candidates;  thr in (0, 1);  k in 1 .. 16384
 *   out_pvalid device [n] fp32;  out_perf device [n] fp32
 *   out_topk   device [k] int64
 * Needs models V and P loaded with the current F (MLT_ENOMODEL otherwise).
 * Asynchronous on `stream`; uses library scratch sized by n (allocated on
 * first use or growth). */
int mlt_screen(void *stream, const float *feats, int64_t n, float thr, int k,
               float *out_pvalid, float *out_perf, int64_t *out_topk);

/* mlt_screen for callers that cannot allocate device memory during a call:
 * a process whose device memory is owned by another allocator (a
 * framework's caching allocator, or a pool reserved up front), or a
 * latency-critical loop that cannot afford cudaMalloc's implicit device
 * synchronisation.  The paper has no counterpart; this is a property of the
 * library only.  Same arguments, results and asynchrony as mlt_screen, but
 * its scratch is a fixed array in the library's own device memory (about
 * 5.1 MB, present on every GPU that loads the library until the process
 * exits), so the call allocates nothing:
 *   - n is limited to 262,144 candidates; a larger n returns MLT_EINVAL
 *     before any GPU work;
 *   - the first call on each device looks up the array's device address on
 *     that device (make it the current device); issue that first call
 *     before any stream capture;
 *   - every call shares the one array: calls whose GPU work overlaps (for
 *     example on two streams without ordering) race and give undefined
 *     results;
 *   - each call clears the array's selection state before its kernels
 *     run, so a call that stopped part-way leaves nothing behind for the
 *     next one;
 *   - a device-side error bit (a bounded wait that gave up) lives in the
 *     array too; mlt_sync_status on the same device reports it (as for the
 *     other entry points) and clears it.  A call that met such an error
 *     leaves its outputs undefined.
 * Models V and P must have been loaded with mlt_load_ensemble beforehand. */
int mlt_screen_noalloc(void *stream, const float *feats, int64_t n, float thr, int k,
                       float *out_pvalid, float *out_perf, int64_t *out_topk);

/* mlt_screen with host buffers, for end-to-end use: copies feats_host
 * ([n][F] fp32) to the device, screens, and copies the three results back
 * into host buffers of the same shapes.  Synchronous on `stream`. */
int mlt_screen_host(void *stream, const float *feats_host, int64_t n, float thr, int k,
                    float *pvalid_host, float *perf_host, int64_t *topk_host);

/* mlt_screen over n_batches independent host batches of n candidates each,
 * pipelined: batch b is screened on `stream` while a library-owned copy
 * stream returns batch b-1's results and uploads batch b+1 (two device
 * staging sets in turn).  Each batch's results are exactly mlt_screen's.
 *   feats_host[b]   host [n][F] fp32 (page-locked memory lets the copies
 *                   overlap the screening)
 *   pvalid_host, perf_host: NULL, or arrays of n_batches host pointers to
 *                   [n] fp32 (a NULL entry skips that batch's copy)
 *   topk_host[b]    host [k] int64
 * The pointer arrays are read during the call only.  Synchronous: returns
 * when every result is on the host. */
int mlt_screen_host_batches(void *stream, int64_t n_batches, const float *const *feats_host, int64_t n,
                            float thr, int k, float *const *pvalid_host, float *const *perf_host,
                            int64_t *const *topk_host);

/* Batched accumulation (Sec. 2: the explorer applies models P and V until
 * it has accumulated (alpha+1)N configurations): candidates 0 .. n_total-1
 * are screened in consecutive batches of `batch`; after each batch the
 * device adds the batch's valid candidates to a running count, and once
 * that count reaches `target` every later batch is skipped on the device
 * (all batches are enqueued up front; no host round trip per batch).
 * out_topk = the k best valid candidates over every batch screened, by the
 * same order as mlt_screen -- identical to mlt_screen over the consumed
 * prefix [0, consumed).
 *   feats      device [n_total][F] fp32
 *   batch >= 1 (at most 65536 batches);  target >= 1
 *   out_pvalid, out_perf: device [n_total] fp32 or NULL; entries of the
 *              consumed prefix are written, later ones are left untouched
 *   out_topk   device [k] int64
 *   out_stats  device int64[3] or NULL: {consumed candidates, valid
 *              candidates kept, batches screened}
 * Asynchronous on `stream`. */
int mlt_screen_until(void *stream, const float *feats, int64_t n_total, int64_t batch,
                     int64_t target, float thr, int k, float *out_pvalid, float *out_perf,
                     int64_t *out_topk, int64_t *out_stats);

/* mlt_screen_until over decoded candidates first_index .. first_index +
 * n_total - 1 of a knob space (see mlt_decode_knobs); out_topk holds
 * candidate indices. */
int mlt_screen_until_decoded(void *stream, const int32_t *radices, const float *option_values,
                             int n_knobs, const mlt_feat_op *program, int64_t first_index,
                             int64_t n_total, int64_t batch, int64_t target, float thr, int k,
                             float *out_pvalid, float *out_perf, int64_t *out_topk,
                             int64_t *out_stats);

/* Explorer proposal step (Sec. 2, "Configuration Explorer": the explorer
 * searches the knob space for configurations the models rank highest; the
 * paper leaves the search open, and this call is one simulated-annealing
 * move of m independent chains, TVM-style).  For chain i:
 *   parent[i] < 0 or >= the size of the space: inactive (next = parent,
 *     score copied, not accepted; an index past the space is also reported
 *     by mlt_sync_status as MLT_EINVAL);
 *   otherwise knob j = knob_draw[i] mod n_knobs of the parent is set to
 *     option index digit_draw[i] mod r_j, giving proposal q;
 *   q is screened like any candidate: s = margin_P(q) if valid, else -inf;
 *   accepted iff s > -inf and fl(s - parent_score[i]) >= fl(temperature *
 *     log_u[i]) (Metropolis: log_u[i] = ln of a uniform draw);
 *   out_next[i] = accepted ? q : parent[i];
 *   out_next_score[i] = accepted ? s : parent_score[i].
 * The random words knob_draw, digit_draw and log_u are the caller's
 * (device [m] uint32, uint32, fp32), so results are reproducible.
 * Decoder arguments as for mlt_decode_knobs (program length = F); models V
 * and P must be loaded.  parent, parent_score, outputs: device [m].
 * temperature > 0; thr in (0, 1).  Asynchronous on `stream`. */
int mlt_sa_step(void *stream, const int32_t *radices, const float *option_values, int n_knobs,
                const mlt_feat_op *program, const int64_t *parent, const float *parent_score,
                const uint32_t *knob_draw, const uint32_t *digit_draw, const float *log_u,
                int64_t m, float temperature, float thr, int64_t *out_next,
                float *out_next_score, int32_t *out_accepted);

/* Cross-rank merge of kept candidates (Sec. 2: the explorer keeps the
 * (alpha+1)N configurations model P ranks highest; with the batch sharded
 * over G ranks, each rank's top-k is gathered and merged): writes to
 * out_topk the k best of the m pairs (scores[i], indices[i]) by the
 * screening's own order -- P score descending (-0 equal to +0), then
 * global candidate index ascending -- padded with -1.
 *   scores   device [m] fp32 (finite for a kept candidate)
 *   indices  device [m] int64 global candidate indices; a negative index
 *            marks an empty slot (ignored); the others must be distinct
 *   m        0 .. 262,144 (for example G ranks x k)
 *   k        1 .. 16,384
 *   out_topk device [k] int64
 * Asynchronous on `stream`. */
int mlt_merge_topk(void *stream, const float *scores, const int64_t *indices, int64_t m, int k,
                   int64_t *out_topk);

/* Model A rerank (Sec. 2, "Hidden Feature Extractor & ML Model A"): from the
 * (alpha+1)N candidates kept by screening, model A -- a performance
 * regressor over visible and hidden features, typically deeper than P
 * (depth 14 in Table 3) -- selects the final N:
 *   out_score[i] = margin_A(row cand[i] of feats) (fp32, tree order) for
 *                  0 <= cand[i] < n; -infinity for cand[i] < 0 (an empty
 *                  slot, e.g. the -1 padding of out_topk);
 *   out_final[r] = the r-th entry of cand by (score descending, candidate
 *                  index ascending), r < n_final; -1 past the valid entries.
 * Arguments:
 *   feats      device [n][F] fp32, the same matrix the candidates index
 *   cand       device [m] int64 (typically mlt_screen's out_topk), 0 <= m <= 16384
 *   n_final    1 .. 16384;  out_score device [m] fp32;  out_final device [n_final] int64
 * Needs model A loaded with the current F.  An index >= n is scored -inf and
 * reported by the next mlt_sync_status (MLT_EINVAL).  Asynchronous. */
int mlt_rerank(void *stream, const float *feats, int64_t n, const int64_t *cand, int m,
               int n_final, float *out_score, int64_t *out_final);

/* Decode candidate indices into knob choices and build their features
 * (the explorer's enumeration of the search space, Sec. 2; knobs are tiling
 * sizes and virtual-thread counts, Appendix A.2; derived features after
 * Table 5).  Candidate i (first_index <= i < first_index + n) is the
 * mixed-radix number with digit j = floor(i / prod_{l<j} r_l) mod r_j, knob
 * 0 least significant; knob j takes option_values[off_j + digit_j] with
 * off_j = r_0 + ... + r_{j-1}.  Feature f is program[f] evaluated on the
 * knob values and the features before it.
 *   radices       host [n_knobs], each 1 .. 256;  n_knobs 1 .. 16;
 *                 sum of radices <= 256
 *   option_values host, the concatenated option tables
 *   program       host [F] instructions, 1 <= F <= 256
 *   first_index + n <= product of the radices
 *   out_knobs     device [n][n_knobs] uint8 option indices, or NULL
 *   out_feats     device [n][F] fp32, or NULL
 * Asynchronous on `stream`. */
int mlt_decode_knobs(void *stream, const int32_t *radices, const float *option_values,
                     int n_knobs, const mlt_feat_op *program, int F, int64_t first_index,
                     int64_t n, uint8_t *out_knobs, float *out_feats);

/* mlt_screen over decoded candidates first_index .. first_index+n-1: the
 * features are built on chip inside the screening kernels and never stored
 * (below the compiled-program threshold, see mlt_tune_decode_jit).
 * The program length must equal the current F.  out_topk holds candidate
 * indices (first_index + position).  Batches of at least the
 * mlt_tune_decode_jit threshold instead build their rows once with the
 * compiled feature program and screen them (same results).  Asynchronous on
 * `stream`. */
int mlt_screen_decoded(void *stream, const int32_t *radices, const float *option_values,
                       int n_knobs, const mlt_feat_op *program, int64_t first_index,
                       int64_t n, float thr, int k, float *out_pvalid, float *out_perf,
                       int64_t *out_topk);

/* Compiled feature program (no counterpart in the paper's text; an
 * implementation choice for decoded screening).  Inside the walk kernels
 * the feature program is interpreted one operation at a time.  For a
 * decoded batch of at least min_n candidates (mlt_screen_decoded, and the
 * proposals of mlt_sa_step; mlt_screen_until_decoded keeps the interpreter)
 * the library instead generates CUDA C from the program
 * -- one statement per feature, the same correctly rounded operation as the
 * interpreter, constants as exact bit patterns -- compiles it with NVRTC
 * once per program and device (the first such call pays the compilation,
 * tens to hundreds of milliseconds), runs it to write the batch's rows
 * [n][F] into a library-owned device buffer (n x F x 4 bytes, grown as
 * needed and kept until exit), and screens those rows.  Results are
 * bit-identical to the interpreted path; only the time differs.  Where
 * NVRTC (libnvrtc.so.13) or the driver library cannot be loaded, the
 * compilation fails or the row buffer cannot be allocated, the call keeps
 * the interpreted path.
 *   min_n   0 (never compile) or the smallest batch that uses it; the
 *           default is 1,048,576
 * mlt_decode_jit_available: 1 if NVRTC and the driver library load.
 * mlt_decode_jit_calls: screening calls so far that ran the compiled
 * program.  Host-only. */
int mlt_tune_decode_jit(int64_t min_n);
int mlt_decode_jit_available(void);
int64_t mlt_decode_jit_calls(void);

/* Wait for `stream` and report errors its queued library work met on the
 * device (MLT_ETIMEOUT for a bounded wait that gave up), clearing them. */
int mlt_sync_status(void *stream);

/* Failure-detection self-test: launches one CTA on `stream` that waits on
 * a shared-memory barrier nothing completes.  The bounded wait every walk
 * kernel uses gives up after limit_ns (1e6 .. 2e9 ns), records the
 * timeout and returns, so the next mlt_sync_status(stream) reports
 * MLT_ETIMEOUT and the device stays usable.  No fault, trap or endless
 * loop is involved.  Asynchronous. */
int mlt_selftest_wait_timeout(void *stream, int64_t limit_ns);

/* Failure-detection self-test inside the screening path: arms a one-shot
 * so that the next screening call whose model V has a full table (depth
 * <= 10) makes V-pass CTA `cta` (clamped to the last CTA) wait for its
 * first tree chunk on a barrier phase that nothing completes.  That wait
 * gives up after limit_ns (1e6 .. 2e9 ns); the CTA lets its copies land,
 * records the timeout, and still completes its tile's bookkeeping (none of
 * its candidates valid), so the call's other results stay consistent and
 * the next call is unaffected.  mlt_sync_status then reports MLT_ETIMEOUT.
 * No fault, trap or endless loop is involved.  Host-only bookkeeping. */
int mlt_selftest_walk_timeout(int cta, int64_t limit_ns);

/* Test support: writes `value` into the four counters (survivor count,
 * collected keys, two CTA tickets) of the selection state that the
 * allocating entry points (static_scratch = 0) or mlt_screen_noalloc
 * (static_scratch != 0) use on the current device, as a call that stopped
 * part-way could leave them.  Every screening call clears that state before
 * its kernels run, so results must not change.  Synchronous. */
int mlt_selftest_poison_state(int static_scratch, uint32_t value);

/* Number of valid candidates found by the last screening call (waits for
 * `stream`). */
int mlt_last_survivor_count(void *stream, int64_t *count_out);

/* Measurement support.  mlt_profile_phases(1) makes every later screening
 * call record CUDA events between its phases on the caller's stream (and
 * clears earlier records); mlt_profile_phases(0) stops recording.  Host-only
 * bookkeeping plus event records; results are unchanged. */
int mlt_profile_phases(int enable);

/* Measurement support: the walk-rate ceiling of a full-table model (depth
 * <= 10) on this batch.  One launch stages tiles of the candidates
 * feats[0, n) (device, [n][F] fp32, as for mlt_screen) the way the V pass
 * does, copies the first R trees of model `model_id`'s table into shared
 * memory once (R = the trees the V-pass shape keeps in its chunk buffers,
 * at most the model's), and walks those R trees `rounds` times per
 * candidate: the screening walk's node test and layout without its chunk
 * streaming.  out_sums[i] (device, [n]) receives the fp32 sum, in walk order,
 * of the rounds x R leaves candidate i reaches (trees 0..R-1, repeated);
 * *visits_out receives the node visits of the launch (n x R x depth x
 * rounds).  The caller times the launch with events on `stream`.
 * Asynchronous; MLT_EINVAL for a bad argument, a compact table or a half
 * table; MLT_ENOMODEL if the model is not loaded for the current F. */
int mlt_walk_peak(void *stream, int model_id, const float *feats, int64_t n, int rounds, float *out_sums,
                  int64_t *visits_out);

/* Waits for the recorded events, then writes for each phase the device time
 * summed over the recorded calls, in ms: out_ms[0] V pass, [1] survivor
 * compaction, [2] P pass, [3] top-k (n_phases <= 4 entries written).
 * *n_calls_out receives the number of recorded calls.  Clears the records. */
int mlt_phase_times(float *out_ms, int n_phases, int64_t *n_calls_out);

/* Tuning: fix the launch shape of the tree walk over model `model_id`'s
 * trees (0 in any field = let the library choose it):
 *   candidates   candidates per CTA: a multiple of 32, 32 .. 384 (above
 *                256 only for fp32 tables of depth <= 10 walked by one
 *                group of warps; 32 .. 256 otherwise)
 *   splits       threads sharing one candidate's trees: 1, 2 or 4 for
 *                ensembles of depth <= 10, 1, 2, 4 or 8 for split tables
 *                (groups of warps, leaves summed in tree order through
 *                shared memory), 1, 2, 4 or 8 for compact tables (lanes of
 *                a warp, summed through shuffles); candidates x splits <=
 *                256 (384 with splits 1 for fp32 tables of depth <= 10,
 *                512 for split tables, 1,024 with 8 groups)
 *   group        trees a thread walks at once: 2, 4 or 8 (depth <= 10 and
 *                split tables), 4 or 8 (compact tables)
 *   chunk_trees  trees per shared-memory chunk: 1, 2, 4, 8 or 16 (full,
 *                half and split tables), 32 (split tables)
 *   nbuf         chunk buffers, 2 or 3 (full, half and split tables)
 * A shape that does not fit shared memory falls back to the library's
 * choice.  Results never depend on the shape.  Host-only. */
int mlt_tune_walk(int model_id, int candidates, int splits, int group, int chunk_trees, int nbuf);

/* Measurement: the launch shape the tree walk over model `model_id`'s
 * trees (V or P, loaded on the current device) would use for a screening
 * call of n candidates -- the V pass (p_pass = 0) walks n, the P pass
 * (p_pass != 0) is planned for about half of them -- including any shape
 * fixed by mlt_tune_walk.  out[7]: candidates per CTA, splits (tree groups
 * or lanes per candidate), trees in flight per thread, trees per chunk,
 * chunk buffers, CTAs resident per SM, table kind (0 full, 1 compact,
 * 2 half, 3 split).  Batches that mlt_screen screens in one launch
 * (mlt_tune_fused_small) do not use this shape.  Host-only. */
int mlt_walk_shape(int model_id, int64_t n, int p_pass, int32_t *out);

/* Tuning: batches of up to max_n candidates (0 .. 8,192; the default is
 * 8,192) with stored features, whose V and P are full tables (depth <= 10)
 * of the same depth small enough to share a CTA's shared memory, are
 * screened by one kernel launch (V walk, validity, P walk, keys and the
 * top-k selection by its last CTA) instead of four; 0 turns that path off.
 * Results never depend on the path.  Host-only. */
int mlt_tune_fused_small(int max_n);

/* Tuning: the table format of models V and P deeper than 10 levels, for
 * ensembles loaded after this call.  levels = 6 (the default) or 7: a
 * split table, whose first `levels` levels stream through shared memory
 * with the tile while the deeper nodes are read from L2; 0: a compact
 * table, read wholly through L1/L2.  Model A always uses the compact
 * table.  Results never depend on the format.  Host-only. */
int mlt_tune_head_levels(int levels);

/* Cumulative number of GPU kernels this library has launched. */
int64_t mlt_kernel_launches(void);

/* Message for the last failing call on this thread ("" if none). */
const char *mlt_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* MLT_H */
