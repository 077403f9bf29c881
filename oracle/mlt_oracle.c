/*
 * mlt_oracle.c -- plain, slow, single-threaded CPU oracle for ML^2Tuner's
 * batched candidate screening (V filter -> P score -> top-k).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or
 * calls this file: only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header, table or helper with the
 * CUDA library; the only thing both sides see is the seeded input data.
 *
 * What it follows (ML^2Tuner, arXiv 2411.10764):
 *   - Sec. 2 "Configuration Explorer": the explorer enumerates the search
 *     space of configurations and scores them with the ML models.  The
 *     mixed-radix decoding of a candidate index into knob choices is this
 *     enumeration written out (orc_decode / orc_features).
 *   - Sec. 2 "ML Model V": validity predicted from the same features as P; a
 *     candidate predicted invalid is never profiled (orc_screen_rows: valid).
 *   - Sec. 2 "ML Model P" and "Hidden Feature Extractor & ML Model A": the
 *     (alpha+1)N kept candidates are those ranked highest by P's predicted
 *     performance (orc_topk).
 *   - Sec. 3 "Experimental Setup" and Appendix A.3 (Table 3): all models are
 *     XGBoost gradient-boosted tree ensembles; a prediction is the sum over
 *     trees of the one leaf each tree routes the feature vector to
 *     (orc_tree_leaf / orc_margin).
 *
 * Readings where the paper is silent (each one is listed in the design notes):
 *   - split rule: go left iff x < threshold; x >= threshold goes right;
 *     a NaN feature (missing value) takes the node's default direction;
 *   - no base score: margin = sum of leaves, accumulated in fp32 in tree
 *     order starting from 0.0f;
 *   - validity: sigmoid(margin_V) >= thr, decided exactly (orc_tau gives the
 *     smallest float margin that passes); with thr = 0.5 this is the sign rule
 *     of the paper's binary:hinge objective (Table 3);
 *   - rank: descending P score, equal scores (-0 == +0) by ascending index;
 *     fewer than k survivors -> the remaining slots hold -1.
 *
 * Build: gcc -O2 -std=c99 -ffp-contract=off -fno-fast-math -shared -fPIC
 * (no fused multiply-add anywhere: every float operation is rounded once).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* One tree slot in implicit heap order: children of slot j are 2j+1, 2j+2.
 * feature >= 0: split on that feature at `value`; -1: leaf with `value`;
 * -2: unused slot.  12 bytes, the documented input layout. */
typedef struct {
    int32_t feature;
    float value;
    uint8_t default_left;
    uint8_t pad[3];
} orc_node;

/* Feature-program instruction (16 bytes, the documented input layout). */
typedef struct {
    int32_t op;
    int32_t a;
    int32_t b;
    float c;
} orc_feat_op;

/* ------------------------------------------------------------------ */
/* Tree-ensemble prediction (Sec. 3 setup: XGBoost gbtree models)     */
/* ------------------------------------------------------------------ */

/* Walk one tree from the root to a leaf and return the leaf value.
 * Returns NaN if the walk leaves the tree (malformed input). */
float orc_tree_leaf(const orc_node *tree, int depth, const float *x)
{
    int64_t slots = ((int64_t)2 << depth) - 1;
    int64_t j = 0;
    for (;;) {
        if (j >= slots)
            return NAN;
        const orc_node *nd = &tree[j];
        if (nd->feature == -1)
            return nd->value;
        if (nd->feature < 0)
            return NAN;
        float v = x[nd->feature];
        int go_left;
        if (isnan(v))
            go_left = nd->default_left != 0;
        else
            go_left = v < nd->value;
        j = go_left ? 2 * j + 1 : 2 * j + 2;
    }
}

/* Ensemble margin: sum of one leaf per tree, fp32, tree 0 first. */
float orc_margin(const orc_node *nodes, int n_trees, int depth, const float *x)
{
    int64_t slots = ((int64_t)2 << depth) - 1;
    float acc = 0.0f;
    for (int t = 0; t < n_trees; ++t) {
        float leaf = orc_tree_leaf(nodes + (int64_t)t * slots, depth, x);
        acc = acc + leaf;
    }
    return acc;
}

/* Margins of rows [0, n) of a row-major [n][F] feature matrix. */
void orc_margins(const orc_node *nodes, int n_trees, int depth,
                 const float *feats, int64_t n, int F, float *out)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = orc_margin(nodes, n_trees, depth, feats + i * (int64_t)F);
}

/* ------------------------------------------------------------------ */
/* Validity decision (Sec. 2 "ML Model V")                            */
/* ------------------------------------------------------------------ */

/* sigmoid(m) >= thr, decided without cancellation:
 *   1/(1+e^-m) >= thr  <=>  e^-m <= (1-thr)/thr  <=>  -m <= log1p((1-2 thr)/thr).
 * 1-2thr is exact in long double for a float thr, so the right-hand side
 * carries only long-double relative rounding error. */
static int passes(float m, float thr)
{
    long double rhs = log1pl((1.0L - 2.0L * (long double)thr) / (long double)thr);
    return -(long double)m <= rhs;
}

/* Map a float to an integer that orders like the float (NaN excluded). */
static int64_t float_order_key(float f)
{
    uint32_t u;
    memcpy(&u, &f, 4);
    if (u & 0x80000000u)
        return -(int64_t)(u & 0x7FFFFFFFu);
    return (int64_t)u;
}

static float float_from_order_key(int64_t k)
{
    uint32_t u = k < 0 ? ((uint32_t)(-k) | 0x80000000u) : (uint32_t)k;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

/* Smallest float m with sigmoid(m) >= thr, for 0 < thr < 1: found by
 * bisection over the ordered float lattice (the predicate is monotone).
 * Returns NaN when thr is outside (0, 1). */
float orc_tau(float thr)
{
    if (!(thr > 0.0f && thr < 1.0f))
        return NAN;
    int64_t lo = float_order_key(-INFINITY); /* sigmoid(-inf) = 0 < thr  */
    int64_t hi = float_order_key(INFINITY);  /* sigmoid(+inf) = 1 >= thr */
    while (hi - lo > 1) {
        int64_t mid = lo + (hi - lo) / 2;
        if (passes(float_from_order_key(mid), thr))
            hi = mid;
        else
            lo = mid;
    }
    float t = float_from_order_key(hi);
    return t == 0.0f ? 0.0f : t; /* -0 and +0 decide alike; report +0 */
}

/* Reported validity probability: sigmoid in double, rounded to float. */
float orc_sigmoid(float m)
{
    return (float)(1.0 / (1.0 + exp(-(double)m)));
}

/* Per-row part of the screening pass for rows [0, n):
 *   pvalid[i] = sigmoid(margin_V(x_i))
 *   valid[i]  = sigmoid(margin_V(x_i)) >= thr   (as margin_V >= tau)
 *   perf[i]   = margin_P(x_i) if valid, -inf otherwise.
 * margin_v (optional, may be NULL) receives margin_V.  Returns 0, or -1 for
 * a threshold outside (0, 1). */
int orc_screen_rows(const float *feats, int64_t n, int F,
                    const orc_node *v_nodes, int v_trees, int v_depth,
                    const orc_node *p_nodes, int p_trees, int p_depth,
                    float thr, float *out_pvalid, float *out_perf,
                    uint8_t *out_valid, float *out_margin_v)
{
    float tau = orc_tau(thr);
    if (isnan(tau))
        return -1;
    for (int64_t i = 0; i < n; ++i) {
        const float *x = feats + i * (int64_t)F;
        float mv = orc_margin(v_nodes, v_trees, v_depth, x);
        int valid = mv >= tau;
        if (out_margin_v)
            out_margin_v[i] = mv;
        out_pvalid[i] = orc_sigmoid(mv);
        out_valid[i] = (uint8_t)valid;
        out_perf[i] = valid ? orc_margin(p_nodes, p_trees, p_depth, x) : -INFINITY;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Top-k by P (Sec. 2 "Hidden Feature Extractor & ML Model A")        */
/* ------------------------------------------------------------------ */

typedef struct {
    float score;
    int64_t index;
} scored;

static int by_score_desc_index_asc(const void *pa, const void *pb)
{
    const scored *a = (const scored *)pa, *b = (const scored *)pb;
    if (a->score > b->score)
        return -1;
    if (a->score < b->score)
        return 1;
    return (a->index > b->index) - (a->index < b->index);
}

/* The k best survivors: full sort of every valid candidate by (score desc,
 * index asc), first k kept; slots past the survivor count hold -1.
 * index_base is added to every emitted index.  Returns the survivor count,
 * or -1 on allocation failure. */
int64_t orc_topk(const float *perf, const uint8_t *valid, int64_t n, int k,
                 int64_t index_base, int64_t *out_topk)
{
    int64_t s = 0;
    for (int64_t i = 0; i < n; ++i)
        s += valid[i] != 0;
    scored *all = (scored *)malloc((size_t)(s > 0 ? s : 1) * sizeof(scored));
    if (!all)
        return -1;
    int64_t w = 0;
    for (int64_t i = 0; i < n; ++i)
        if (valid[i]) {
            all[w].score = perf[i];
            all[w].index = i;
            ++w;
        }
    qsort(all, (size_t)s, sizeof(scored), by_score_desc_index_asc);
    for (int r = 0; r < k; ++r)
        out_topk[r] = r < s ? all[r].index + index_base : -1;
    free(all);
    return s;
}

/* Whole screening pass over rows [0, n): per-row part, then top-k. */
int64_t orc_screen(const float *feats, int64_t n, int F,
                   const orc_node *v_nodes, int v_trees, int v_depth,
                   const orc_node *p_nodes, int p_trees, int p_depth,
                   float thr, int k, float *out_pvalid, float *out_perf,
                   int64_t *out_topk)
{
    uint8_t *valid = (uint8_t *)malloc((size_t)(n > 0 ? n : 1));
    if (!valid)
        return -1;
    if (orc_screen_rows(feats, n, F, v_nodes, v_trees, v_depth, p_nodes,
                        p_trees, p_depth, thr, out_pvalid, out_perf, valid,
                        NULL) != 0) {
        free(valid);
        return -1;
    }
    int64_t s = orc_topk(out_perf, valid, n, k, 0, out_topk);
    free(valid);
    return s;
}

/* ------------------------------------------------------------------ */
/* Model A rerank (Sec. 2 "Hidden Feature Extractor & ML Model A")     */
/* ------------------------------------------------------------------ */

/* From the kept candidates cand[0..m), model A -- a performance regressor
 * over visible and hidden features -- selects the final n_final:
 *   out_score[i] = margin_A(feats row cand[i]) for cand[i] >= 0, -inf else;
 *   out_final    = the n_final entries of cand with the highest score, equal
 *                  scores by the smaller candidate index, -1 padded.
 * Returns the number of valid entries, or -1 on allocation failure. */
int64_t orc_rerank(const float *feats, int F, const int64_t *cand, int64_t m,
                   const orc_node *a_nodes, int a_trees, int a_depth, int n_final,
                   float *out_score, int64_t *out_final)
{
    scored *all = (scored *)malloc((size_t)(m > 0 ? m : 1) * sizeof(scored));
    if (!all)
        return -1;
    int64_t v = 0;
    for (int64_t i = 0; i < m; ++i) {
        if (cand[i] < 0) {
            out_score[i] = -INFINITY;
            continue;
        }
        float s = orc_margin(a_nodes, a_trees, a_depth, feats + cand[i] * (int64_t)F);
        out_score[i] = s;
        all[v].score = s;
        all[v].index = cand[i];
        ++v;
    }
    qsort(all, (size_t)v, sizeof(scored), by_score_desc_index_asc);
    for (int r = 0; r < n_final; ++r)
        out_final[r] = r < v ? all[r].index : -1;
    free(all);
    return v;
}

/* ------------------------------------------------------------------ */
/* Knob decoding and feature program (Sec. 2 "Configuration Explorer") */
/* ------------------------------------------------------------------ */

/* Mixed-radix decode of candidate indices first .. first+n-1 into one
 * option index per knob, knob 0 least significant:
 *   digit_j(i) = floor(i / prod_{l<j} r_l) mod r_j.
 * out_digits is [n][n_knobs].  Returns 0, or -1 if an index is beyond the
 * size of the space. */
int orc_decode(const int32_t *radices, int n_knobs, int64_t first, int64_t n,
               uint8_t *out_digits)
{
    long double space = 1.0L;
    for (int j = 0; j < n_knobs; ++j)
        space *= (long double)radices[j];
    if ((long double)first + (long double)n > space)
        return -1;
    for (int64_t r = 0; r < n; ++r) {
        int64_t rem = first + r;
        for (int j = 0; j < n_knobs; ++j) {
            out_digits[r * n_knobs + j] = (uint8_t)(rem % radices[j]);
            rem /= radices[j];
        }
    }
    return 0;
}

static float ilog2_exact(float a)
{
    if (!(a > 0.0f) || !isnormal(a) || isinf(a))
        return 0.0f;
    int e;
    frexpf(a, &e); /* a = m * 2^e with m in [0.5, 1) */
    return (float)(e - 1);
}

/* One operand: -1 -> the constant c; [0, n_knobs) -> that knob's option
 * value; n_knobs + f -> feature f of this row (f below the one computed). */
static float operand(int32_t s, float c, const float *knob_val, int n_knobs,
                     const float *row)
{
    if (s == -1)
        return c;
    if (s < n_knobs)
        return knob_val[s];
    return row[s - n_knobs];
}

/* Evaluate the feature program for one decoded candidate.  Every operation
 * is a single IEEE-754 single-precision operation, rounded to nearest. */
static int run_program(const orc_feat_op *prog, int F, const float *knob_val,
                       int n_knobs, float *row)
{
    for (int i = 0; i < F; ++i) {
        const orc_feat_op *o = &prog[i];
        if (o->a < -1 || o->a >= n_knobs + i || o->b < -1 || o->b >= n_knobs + i)
            return -1;
        float A = operand(o->a, o->c, knob_val, n_knobs, row);
        float B = operand(o->b, o->c, knob_val, n_knobs, row);
        float x;
        switch (o->op) {
        case 0: x = A; break;                              /* COPY    */
        case 1: x = ilog2_exact(A); break;                 /* ILOG2   */
        case 2: x = A + B; break;                          /* ADD     */
        case 3: x = A - B; break;                          /* SUB     */
        case 4: x = A * B; break;                          /* MUL     */
        case 5: x = A / B; break;                          /* DIV     */
        case 6: { float q = A / B; x = ceilf(q); } break;  /* CEILDIV */
        case 7: {                                          /* REM     */
            float q = A / B;
            float fq = floorf(q);
            float p = B * fq;
            x = A - p;
        } break;
        case 8: x = (B < A) ? B : A; break;                /* MIN     */
        case 9: x = (B > A) ? B : A; break;                /* MAX     */
        case 10: x = (A > B) ? 1.0f : 0.0f; break;         /* GT      */
        case 11: x = (A == B) ? 1.0f : 0.0f; break;        /* EQ      */
        default: return -1;
        }
        row[i] = x;
    }
    return 0;
}

/* Decode candidates first .. first+n-1 and build their feature rows.
 * option_values holds, knob after knob, r_j option values for knob j.
 * out_knobs ([n][n_knobs] option indices) may be NULL; out_feats is [n][F].
 * Returns 0, or -1 on an index beyond the space or a malformed program. */
int orc_features(const int32_t *radices, const float *option_values,
                 int n_knobs, const orc_feat_op *program, int F, int64_t first,
                 int64_t n, uint8_t *out_knobs, float *out_feats)
{
    if (n_knobs <= 0 || n_knobs > 64)
        return -1;
    uint8_t digits[64];
    float knob_val[64];
    int32_t offset[64];
    int32_t off = 0;
    for (int j = 0; j < n_knobs; ++j) {
        if (radices[j] <= 0 || radices[j] > 256)
            return -1;
        offset[j] = off;
        off += radices[j];
    }
    for (int64_t r = 0; r < n; ++r) {
        if (orc_decode(radices, n_knobs, first + r, 1, digits) != 0)
            return -1;
        for (int j = 0; j < n_knobs; ++j) {
            knob_val[j] = option_values[offset[j] + digits[j]];
            if (out_knobs)
                out_knobs[r * n_knobs + j] = digits[j];
        }
        if (run_program(program, F, knob_val, n_knobs, out_feats + r * (int64_t)F) != 0)
            return -1;
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Explorer proposal step (Sec. 2 "Configuration Explorer")           */
/* ------------------------------------------------------------------ */

/* One simulated-annealing step over m chains of the knob space.  The paper
 * leaves the explorer's search unspecified beyond "selects configurations
 * with the highest potential"; this step is the build's reading:
 *   chain i with parent[i] < 0 is inactive (next = parent, score copied);
 *   otherwise knob j = knob_draw[i] mod n_knobs of the parent is set to
 *   digit d = digit_draw[i] mod r_j, giving proposal q;
 *   q is scored like any candidate: s = margin_P(q) if V finds it valid
 *   (sigmoid(margin_V) >= thr), else -inf;
 *   accept iff s > -inf and fl(s - parent_score[i]) >= fl(temperature *
 *   log_u[i])  (Metropolis with the log of a uniform draw passed in);
 *   next = accept ? q : parent, next_score = accept ? s : parent_score.
 * Returns 0, or -1 on a malformed program / threshold. */
int orc_sa_step(const int32_t *radices, const float *option_values, int n_knobs,
                const orc_feat_op *program, int F, const orc_node *v_nodes, int v_trees,
                int v_depth, const orc_node *p_nodes, int p_trees, int p_depth,
                const int64_t *parent, const float *parent_score, const uint32_t *knob_draw,
                const uint32_t *digit_draw, const float *log_u, int64_t m, float temperature,
                float thr, int64_t *out_next, float *out_next_score, int32_t *out_accepted)
{
    float tau = orc_tau(thr);
    if (isnan(tau) || n_knobs <= 0 || n_knobs > 64)
        return -1;
    float *row = (float *)malloc((size_t)(F > 0 ? F : 1) * sizeof(float));
    if (!row)
        return -1;
    int rc = 0;
    for (int64_t i = 0; i < m && rc == 0; ++i) {
        if (parent[i] < 0) {
            out_next[i] = parent[i];
            out_next_score[i] = parent_score[i];
            out_accepted[i] = 0;
            continue;
        }
        /* parent's digits, knob 0 least significant */
        int32_t digit[64];
        int64_t rem = parent[i];
        for (int j = 0; j < n_knobs; ++j) {
            digit[j] = (int32_t)(rem % radices[j]);
            rem /= radices[j];
        }
        int kj = (int)(knob_draw[i] % (uint32_t)n_knobs);
        digit[kj] = (int32_t)(digit_draw[i] % (uint32_t)radices[kj]);
        int64_t q = 0, place = 1;
        for (int j = 0; j < n_knobs; ++j) {
            q += digit[j] * place;
            place *= radices[j];
        }
        uint8_t knobs[64];
        if (orc_features(radices, option_values, n_knobs, program, F, q, 1, knobs, row) != 0) {
            rc = -1;
            break;
        }
        float mv = orc_margin(v_nodes, v_trees, v_depth, row);
        float s = mv >= tau ? orc_margin(p_nodes, p_trees, p_depth, row) : -INFINITY;
        int accept = 0;
        if (s != -INFINITY) {
            float d = s - parent_score[i];
            float bar = temperature * log_u[i];
            accept = d >= bar;
        }
        out_next[i] = accept ? q : parent[i];
        out_next_score[i] = accept ? s : parent_score[i];
        out_accepted[i] = accept;
    }
    free(row);
    return rc;
}
