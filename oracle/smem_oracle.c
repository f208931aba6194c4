/*
 * smem_oracle.c -- fp64 CPU oracle of the SMem reader's attention.
 *
 * TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this file's library.
 * The product path (paper_2609_32395_gb300) never calls it and shares no code
 * with it.
 *
 * What it computes is the plain definition of the reader's two attentions
 * (arXiv 2609.32395, Sec. 2 "Model" and App. A "Reader"):
 *
 *   block-local causal self-attention: a position attends to the positions
 *   of its own block up to and including itself, never across a block
 *   boundary;
 *
 *   cross-attention: every query of block i attends to the memory rows of
 *   the strictly earlier blocks (block index < i, the block-causal mask),
 *   with a learned null row prepended (App. A, "Positions and memory");
 *   the memory is a multiset stored canonically ordered by block index
 *   (Sec. 2, "Model"), which makes reads a function of the block set alone
 *   (Theorem 1).
 *
 * Each attention is a softmax over its key list with scale 1/sqrt(d_h),
 * computed in two passes (maximum, then exponentials and sums) with the C
 * library's exp in fp64, loops in canonical order. An empty key list gives
 * a zero output. Nothing is blocked, fused or reordered beyond that. Heads
 * are independent: built with OpenMP, the per-head loops spread heads over
 * threads, each head computed by one thread in the same order as alone.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_ERR_DUPLICATE (-4)
#define ORACLE_ERR_ALLOC (-12)

/* softmax(scale * q . k_r) weighted sum of v_r over the rows listed in
 * krows/vrows (each a pointer to D doubles), in list order. */
static int attend(int D, double scale, const double *q, long nk,
                  const double *const *krows, const double *const *vrows,
                  double *out)
{
    long r;
    int d;
    double m, den;
    double *s;
    if (nk == 0) {
        for (d = 0; d < D; ++d) out[d] = 0.0;
        return 0;
    }
    s = (double *)malloc(sizeof(double) * (size_t)nk);
    if (!s) return ORACLE_ERR_ALLOC;
    m = -INFINITY;
    for (r = 0; r < nk; ++r) {
        double dot = 0.0;
        for (d = 0; d < D; ++d) dot += q[d] * krows[r][d];
        s[r] = scale * dot;
        if (s[r] > m) m = s[r];
    }
    den = 0.0;
    for (d = 0; d < D; ++d) out[d] = 0.0;
    for (r = 0; r < nk; ++r) {
        double e = exp(s[r] - m);
        den += e;
        for (d = 0; d < D; ++d) out[d] += e * vrows[r][d];
    }
    for (d = 0; d < D; ++d) out[d] /= den;
    free(s);
    return 0;
}

/* Block-causal row-set resolution: the blocks with index < q_idx, in
 * ascending block index. Writes their positions in the given list to
 * order_out and returns how many there are, or ORACLE_ERR_DUPLICATE when a
 * block index occurs twice. Insertion sort: the lists here are short. */
int oracle_rowset(int n_blocks, const int32_t *block_idx, int32_t q_idx,
                  int32_t *order_out)
{
    int i, j, n = 0;
    for (i = 0; i < n_blocks; ++i)
        for (j = i + 1; j < n_blocks; ++j)
            if (block_idx[i] == block_idx[j]) return ORACLE_ERR_DUPLICATE;
    for (i = 0; i < n_blocks; ++i) {
        if (block_idx[i] >= q_idx) continue;
        j = n++;
        while (j > 0 && block_idx[order_out[j - 1]] > block_idx[i]) {
            order_out[j] = order_out[j - 1];
            --j;
        }
        order_out[j] = i;
    }
    return n;
}

/* Cross-attention row pointers for head h: null row (if any), then rows
 * 0..R-1 of each selected block in canonical order. blocks_* are
 * [n_blocks][H][R][D]; null_* are [H][D]. */
static long ca_rows(int H, int R, int D, int h, int n_sel, const int32_t *order,
                    const double *blocks_k, const double *blocks_v,
                    int has_null, const double *k_null, const double *v_null,
                    const double **kr, const double **vr)
{
    long n = 0;
    int i, r;
    if (has_null) {
        kr[n] = k_null + (size_t)h * D;
        vr[n] = v_null + (size_t)h * D;
        ++n;
    }
    for (i = 0; i < n_sel; ++i) {
        size_t base = (((size_t)order[i] * H + h) * R) * D;
        for (r = 0; r < R; ++r) {
            kr[n] = blocks_k + base + (size_t)r * D;
            vr[n] = blocks_v + base + (size_t)r * D;
            ++n;
        }
    }
    return n;
}

/* Threads of the per-head loops below (OpenMP when the library was built
 * with it; each head is computed by one thread exactly as it would be
 * alone, so the result does not depend on the thread count). Returns the
 * thread count in effect. */
int oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}

/* The one-block pass of one head (its own row-pointer lists). */
static int prefill_head(int h, int H, int D, int b, int R, int n_sel, const int32_t *order,
                        const double *blocks_k, const double *blocks_v,
                        int has_null, const double *k_null, const double *v_null, long nrows,
                        const double *qs, const double *ks, const double *vs,
                        const double *qc, double *osa, double *oca)
{
    const double scale = 1.0 / sqrt((double)D);
    const double **kr, **vr;
    int t, u, rc = 0;
    kr = (const double **)malloc(sizeof(double *) * (size_t)(nrows + b + 1));
    vr = (const double **)malloc(sizeof(double *) * (size_t)(nrows + b + 1));
    if (!kr || !vr) { free(kr); free(vr); return ORACLE_ERR_ALLOC; }
    /* self-attention inside the block: query t sees keys 0..t */
    for (t = 0; t < b && rc == 0; ++t) {
        for (u = 0; u <= t; ++u) {
            kr[u] = ks + ((size_t)u * H + h) * D;
            vr[u] = vs + ((size_t)u * H + h) * D;
        }
        rc = attend(D, scale, qs + ((size_t)t * H + h) * D, t + 1, kr, vr,
                    osa + ((size_t)t * H + h) * D);
    }
    /* cross-attention into the rows of strictly earlier blocks */
    ca_rows(H, R, D, h, n_sel, order, blocks_k, blocks_v, has_null, k_null, v_null, kr, vr);
    for (t = 0; t < b && rc == 0; ++t)
        rc = attend(D, scale, qc + ((size_t)t * H + h) * D, nrows, kr, vr,
                    oca + ((size_t)t * H + h) * D);
    free(kr);
    free(vr);
    return rc;
}

/*
 * One-block reader pass for one layer (block-skip serving, Sec. 3.1):
 *   qs, ks, vs, qc: [b][H][D] self-attention Q/K/V and cross-attention Q of
 *   the query block; osa, oca: [b][H][D] outputs.
 *   Memory: n_blocks blocks given in any order, block_idx[n_blocks] their
 *   indices, blocks_k/v [n_blocks][H][R][D].
 * Returns 0, or a negative error.
 */
int oracle_reader_prefill(int H, int D, int b, int R,
                          int n_blocks, const int32_t *block_idx,
                          const double *blocks_k, const double *blocks_v,
                          int has_null, const double *k_null, const double *v_null,
                          int32_t q_idx,
                          const double *qs, const double *ks, const double *vs,
                          const double *qc, double *osa, double *oca)
{
    int32_t *order;
    long nrows;
    int n_sel, h, rc = 0;

    order = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n_blocks > 0 ? n_blocks : 1));
    if (!order) return ORACLE_ERR_ALLOC;
    n_sel = oracle_rowset(n_blocks, block_idx, q_idx, order);
    if (n_sel < 0) { free(order); return n_sel; }
    nrows = (long)n_sel * R + (has_null ? 1 : 0);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (h = 0; h < H; ++h) {
        int r = prefill_head(h, H, D, b, R, n_sel, order, blocks_k, blocks_v, has_null, k_null, v_null,
                             nrows, qs, ks, vs, qc, osa, oca);
        if (r) {
#ifdef _OPENMP
#pragma omp critical
#endif
            rc = r;
        }
    }
    free(order);
    return rc;
}

/* The decode step of one head (its own row-pointer lists). */
static int decode_head(int h, int H, int D, int R, int n_sel, const int32_t *order,
                       const double *blocks_k, const double *blocks_v,
                       int has_null, const double *k_null, const double *v_null, long nrows, int p,
                       const double *kin, const double *vin,
                       const double *qs, const double *k_new, const double *v_new,
                       const double *qc, double *osa, double *oca)
{
    const double scale = 1.0 / sqrt((double)D);
    const double **kr, **vr;
    int u, rc;
    kr = (const double **)malloc(sizeof(double *) * (size_t)(nrows + p + 2));
    vr = (const double **)malloc(sizeof(double *) * (size_t)(nrows + p + 2));
    if (!kr || !vr) { free(kr); free(vr); return ORACLE_ERR_ALLOC; }
    for (u = 0; u < p; ++u) {
        kr[u] = kin + ((size_t)u * H + h) * D;
        vr[u] = vin + ((size_t)u * H + h) * D;
    }
    kr[p] = k_new + (size_t)h * D;
    vr[p] = v_new + (size_t)h * D;
    rc = attend(D, scale, qs + (size_t)h * D, p + 1, kr, vr, osa + (size_t)h * D);
    if (rc == 0) {
        ca_rows(H, R, D, h, n_sel, order, blocks_k, blocks_v, has_null, k_null, v_null, kr, vr);
        rc = attend(D, scale, qc + (size_t)h * D, nrows, kr, vr, oca + (size_t)h * D);
    }
    free(kr);
    free(vr);
    return rc;
}

/*
 * One decode step for one sequence and one layer (KV-cached decode,
 * Sec. 3.1 and App. "Serving measurements"): the new token sits at in-block
 * offset p; its self-attention keys are the p earlier in-block rows
 * kin/vin [p][H][D] followed by its own k_new/v_new [H][D]; its
 * cross-attention rows are as in the one-block pass.
 *   qs, qc: [H][D]; osa, oca: [H][D].
 */
int oracle_reader_decode(int H, int D, int R,
                         int n_blocks, const int32_t *block_idx,
                         const double *blocks_k, const double *blocks_v,
                         int has_null, const double *k_null, const double *v_null,
                         int32_t q_idx, int p,
                         const double *kin, const double *vin,
                         const double *qs, const double *k_new, const double *v_new,
                         const double *qc, double *osa, double *oca)
{
    int32_t *order;
    long nrows;
    int n_sel, h, rc = 0;

    order = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n_blocks > 0 ? n_blocks : 1));
    if (!order) return ORACLE_ERR_ALLOC;
    n_sel = oracle_rowset(n_blocks, block_idx, q_idx, order);
    if (n_sel < 0) { free(order); return n_sel; }
    nrows = (long)n_sel * R + (has_null ? 1 : 0);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (h = 0; h < H; ++h) {
        int r = decode_head(h, H, D, R, n_sel, order, blocks_k, blocks_v, has_null, k_null, v_null, nrows,
                            p, kin, vin, qs, k_new, v_new, qc, osa, oca);
        if (r) {
#ifdef _OPENMP
#pragma omp critical
#endif
            rc = r;
        }
    }
    free(order);
    return rc;
}
