/*
 * A plain C client of libmlt: the screening boundary used without Python.
 *
 *   screen_client check          host-only calls (no GPU needed): argument
 *                                validation and the validity cut
 *   screen_client IN OUT         loads the ensembles and features in IN,
 *                                screens them with mlt_screen_host (host
 *                                buffers only) and writes the results to OUT
 *
 * IN (little-endian): int32 F, int64 n, float thr, int32 k, then for V and P
 * int32 n_trees, int32 depth and n_trees * (2^(depth+1)-1) 12-byte mlt_node
 * slots, then n * F fp32 features.  OUT: n fp32 pvalid, n fp32 perf, k int64
 * top-k.  The exit status is 0 on success, else the failing call's status
 * (made positive).
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "mlt.h"

static int fail(const char *what, int rc) {
    fprintf(stderr, "%s failed (%d): %s\n", what, rc, mlt_last_error());
    return rc < 0 ? -rc : 1;
}

static int check(void) {
    float tau = 1.0f;
    int rc = mlt_validity_cut(0.5f, &tau);
    if (rc != MLT_OK || tau != 0.0f) return fail("mlt_validity_cut(0.5)", rc ? rc : -1);
    if (mlt_validity_cut(1.5f, &tau) != MLT_EINVAL) return fail("mlt_validity_cut(1.5) accepted", -1);
    if (mlt_set_num_features(0) != MLT_EINVAL) return fail("mlt_set_num_features(0) accepted", -1);
    if (mlt_set_num_features(4) != MLT_OK) return fail("mlt_set_num_features(4)", -1);
    mlt_node stump[3];
    memset(stump, 0, sizeof(stump));
    stump[0].feature = 9; /* feature >= F */
    stump[1].feature = -1;
    stump[2].feature = -1;
    if (mlt_load_ensemble(MLT_MODEL_V, stump, 1, 1) != MLT_EINVAL) return fail("bad ensemble accepted", -1);
    if (mlt_screen_host(NULL, NULL, 10, 0.5f, 0, NULL, NULL, NULL) != MLT_EINVAL) return fail("k = 0 accepted", -1);
    printf("check ok\n");
    return 0;
}

static void *read_all(const char *path, size_t *size) {
    FILE *f = fopen(path, "rb");
    if (!f) return NULL;
    fseek(f, 0, SEEK_END);
    long len = ftell(f);
    fseek(f, 0, SEEK_SET);
    void *buf = malloc(len > 0 ? (size_t)len : 1);
    if (buf && fread(buf, 1, (size_t)len, f) != (size_t)len) {
        free(buf);
        buf = NULL;
    }
    fclose(f);
    *size = (size_t)len;
    return buf;
}

int main(int argc, char **argv) {
    if (argc == 2 && strcmp(argv[1], "check") == 0) return check();
    if (argc != 3) {
        fprintf(stderr, "usage: %s check | %s IN OUT\n", argv[0], argv[0]);
        return 2;
    }
    size_t size = 0;
    unsigned char *in = read_all(argv[1], &size);
    if (!in) return 2;
    unsigned char *p = in;
    int32_t F, k;
    int64_t n;
    float thr;
    memcpy(&F, p, 4); p += 4;
    memcpy(&n, p, 8); p += 8;
    memcpy(&thr, p, 4); p += 4;
    memcpy(&k, p, 4); p += 4;
    int rc = mlt_set_num_features(F);
    if (rc != MLT_OK) return fail("mlt_set_num_features", rc);
    for (int model = MLT_MODEL_V; model <= MLT_MODEL_P; ++model) {
        int32_t n_trees, depth;
        memcpy(&n_trees, p, 4); p += 4;
        memcpy(&depth, p, 4); p += 4;
        const size_t slots = (size_t)n_trees * (((size_t)2 << depth) - 1);
        rc = mlt_load_ensemble(model, (const mlt_node *)p, n_trees, depth);
        if (rc != MLT_OK) return fail("mlt_load_ensemble", rc);
        p += slots * sizeof(mlt_node);
    }
    const float *feats = (const float *)p;
    float *pvalid = malloc(sizeof(float) * (size_t)(n > 0 ? n : 1));
    float *perf = malloc(sizeof(float) * (size_t)(n > 0 ? n : 1));
    int64_t *topk = malloc(sizeof(int64_t) * (size_t)k);
    rc = mlt_screen_host(NULL, feats, n, thr, k, pvalid, perf, topk);
    if (rc != MLT_OK) return fail("mlt_screen_host", rc);
    FILE *out = fopen(argv[2], "wb");
    if (!out) return 2;
    fwrite(pvalid, sizeof(float), (size_t)n, out);
    fwrite(perf, sizeof(float), (size_t)n, out);
    fwrite(topk, sizeof(int64_t), (size_t)k, out);
    fclose(out);
    free(pvalid);
    free(perf);
    free(topk);
    free(in);
    return 0;
}
