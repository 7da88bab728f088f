/*
 * ProViP oracle: a plain, slow, fp64 CPU restatement of the token-pruning path
 * of "Not All Attention Heads Contribute to Critical Visual Token Selection:
 * Head-Aware Pruning Matters More" (ProViP).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may link, load or call
 * this file: only the tests, the smoke check and the CPU-baseline leg of the
 * benchmark use it. It shares no code, header, table or helper with the CUDA
 * library; it is written directly from the paper's equations, one function per
 * equation group, with plain loops and no blocking, fusion or reordering.
 *
 * Every floating-point step is double precision. Inputs are whatever values the
 * caller hands in (the tests pass the exact bf16/fp32 values given to the GPU,
 * widened to double).
 *
 * Functions and the passages they follow:
 *   po_crit_text        Sec. 4.2, the ranking criterion r and the set T.
 *   po_relevance        Sec. 4.3, the cosine matrix M, its row de-meaning and
 *                       the max-pooled importance p.
 *   po_topk             Sec. 4.3 (top N1 of p) and Sec. 4.4 (top N2 of v).
 *   po_merge            Sec. 4.3, last paragraph: pruned tokens aggregated
 *                       into their nearest kept centroid. The paper defers the
 *                       rule to ApET and does not state it; this function
 *                       implements the reading "cosine-nearest kept token,
 *                       uniform mean of the centroid and its members".
 *                       PARITY UNPINNED BY THE PAPER: only that reading,
 *                       brute force and invariants pin it.
 *   po_attn_row         Sec. 4.4, one row of the cross-modal attention map
 *                       A^cross (softmax over the full causal key range).
 *   po_head_scores      Sec. 4.4, S^vis (mean over the selected heads) and
 *                       the token importance v (mean over text rows).
 *   po_head_confidence  Sec. 4.4, head confidence C^h (sum over critical text
 *                       rows of the population variance of A^cross rows).
 *   po_compact_map      Sec. 4.1 ("pruned tokens are excluded from all
 *                       subsequent computations"): which input rows survive,
 *                       in order.
 *   po_gather_rows      the compaction itself: a byte-exact row gather.
 *   po_prune_batch      Sec. 4.4 end to end for a batch (head scores, top-k,
 *                       compaction of hidden/K/V/pos), OpenMP over samples;
 *                       used for the timed CPU baseline.
 *
 * Return codes: 0 on success, -1 on an invalid argument, -2 on allocation
 * failure.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double dot_d(const double *a, const double *b, int d) {
    double s = 0.0;
    for (int e = 0; e < d; ++e) s += a[e] * b[e];
    return s;
}

/* ---------------------------------------------------------------------------
 * Sec. 4.2. r = (1/N_t) * sum_i Softmax(E_t E_t^T)_i  (row i of the row-wise
 * softmax, no scaling: the paper writes none), T = { j : r_j > Mean(r) }.
 * E: [n, d] row-major. r: [n]. mask: [n], 1 for j in T.
 * If no r_j exceeds the mean (e.g. n == 1 or all rows equal), T is all rows.
 * ------------------------------------------------------------------------- */
int po_crit_text(const double *E, int n, int d, double *r, uint8_t *mask) {
    if (n <= 0 || d <= 0 || !E || !r || !mask) return -1;
    double *row = (double *)malloc(sizeof(double) * (size_t)n);
    if (!row) return -2;
    for (int j = 0; j < n; ++j) r[j] = 0.0;
    for (int i = 0; i < n; ++i) {
        /* row i of G = E E^T */
        double mx = -INFINITY;
        for (int j = 0; j < n; ++j) {
            row[j] = dot_d(E + (size_t)i * d, E + (size_t)j * d, d);
            if (row[j] > mx) mx = row[j];
        }
        /* softmax along the row */
        double z = 0.0;
        for (int j = 0; j < n; ++j) z += exp(row[j] - mx);
        for (int j = 0; j < n; ++j) r[j] += exp(row[j] - mx) / z;
    }
    for (int j = 0; j < n; ++j) r[j] /= (double)n;
    double mean = 0.0;
    for (int j = 0; j < n; ++j) mean += r[j];
    mean /= (double)n;
    int cnt = 0;
    for (int j = 0; j < n; ++j) {
        mask[j] = (uint8_t)(r[j] > mean);
        cnt += mask[j];
    }
    if (cnt == 0)
        for (int j = 0; j < n; ++j) mask[j] = 1;
    free(row);
    return 0;
}

/* cosine similarity; a zero-norm vector has cosine 0 with everything */
static double cos_d(const double *a, const double *b, int d) {
    double na = sqrt(dot_d(a, a, d)), nb = sqrt(dot_d(b, b, d));
    if (na == 0.0 || nb == 0.0) return 0.0;
    return dot_d(a, b, d) / (na * nb);
}

/* ---------------------------------------------------------------------------
 * Sec. 4.3. For the critical text rows i (mask[i] != 0, ascending) and all
 * visual rows j:
 *   M_ij   = cos(E_t[i], E_v[j])
 *   Mh_ij  = M_ij - (1/N_v) sum_k M_ik
 *   p_j    = max_i Mh_ij
 * Et: [nt, d], Ev: [nv, d]. p: [nv].
 * Optional outputs (may be NULL): M [|T|, nv] and mu [|T|] (the row means).
 * ------------------------------------------------------------------------- */
int po_relevance(const double *Et, const uint8_t *mask, int nt, const double *Ev,
                 int nv, int d, double *p, double *M_out, double *mu_out) {
    if (nt <= 0 || nv <= 0 || d <= 0 || !Et || !mask || !Ev || !p) return -1;
    int nT = 0;
    for (int i = 0; i < nt; ++i) nT += mask[i] != 0;
    if (nT == 0) return -1;
    double *M = (double *)malloc(sizeof(double) * (size_t)nT * nv);
    if (!M) return -2;
    int a = 0;
    for (int i = 0; i < nt; ++i) {
        if (!mask[i]) continue;
        for (int j = 0; j < nv; ++j)
            M[(size_t)a * nv + j] = cos_d(Et + (size_t)i * d, Ev + (size_t)j * d, d);
        ++a;
    }
    for (int j = 0; j < nv; ++j) p[j] = -INFINITY;
    for (a = 0; a < nT; ++a) {
        double mu = 0.0;
        for (int k = 0; k < nv; ++k) mu += M[(size_t)a * nv + k];
        mu /= (double)nv;
        if (mu_out) mu_out[a] = mu;
        for (int j = 0; j < nv; ++j) {
            double mh = M[(size_t)a * nv + j] - mu;
            if (mh > p[j]) p[j] = mh;
        }
    }
    if (M_out) memcpy(M_out, M, sizeof(double) * (size_t)nT * nv);
    free(M);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Top-k (Sec. 4.3 top N1 of p; Sec. 4.4 top N2 of v). The k largest scores,
 * ties broken toward the lower index, returned in ascending index order.
 * Implemented as a library sort by (score descending, index ascending).
 * ------------------------------------------------------------------------- */
typedef struct { double s; int i; } po_key;

static int po_key_cmp(const void *x, const void *y) {
    const po_key *a = (const po_key *)x, *b = (const po_key *)y;
    if (a->s > b->s) return -1;
    if (a->s < b->s) return 1;
    return (a->i > b->i) - (a->i < b->i);
}

static int po_int_cmp(const void *x, const void *y) {
    int a = *(const int *)x, b = *(const int *)y;
    return (a > b) - (a < b);
}

int po_topk(const double *s, int n, int k, int *idx) {
    if (n <= 0 || k < 1 || k > n || !s || !idx) return -1;
    po_key *keys = (po_key *)malloc(sizeof(po_key) * (size_t)n);
    if (!keys) return -2;
    for (int i = 0; i < n; ++i) { keys[i].s = s[i]; keys[i].i = i; }
    qsort(keys, (size_t)n, sizeof(po_key), po_key_cmp);
    for (int a = 0; a < k; ++a) idx[a] = keys[a].i;
    qsort(idx, (size_t)k, sizeof(int), po_int_cmp);
    free(keys);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Sec. 4.3, last paragraph (rule not stated by the paper; reading above).
 * keep: [n1] ascending indices of the retained (centroid) rows.
 * assign: [nv]; assign[j] = a, the position in keep of row j's centroid
 *   (kept rows are their own centroid; a pruned row goes to the kept row of
 *   largest cosine, ties to the lowest position).
 * merged: [n1, d]; merged[a] = (E_v[keep[a]] + sum of its members) / (1 + count).
 * ------------------------------------------------------------------------- */
int po_merge(const double *Ev, int nv, int d, const int *keep, int n1, int *assign,
             double *merged) {
    if (nv <= 0 || d <= 0 || n1 < 1 || n1 > nv || !Ev || !keep || !assign || !merged)
        return -1;
    int *pos = (int *)malloc(sizeof(int) * (size_t)nv);
    int *cnt = (int *)calloc((size_t)n1, sizeof(int));
    if (!pos || !cnt) { free(pos); free(cnt); return -2; }
    for (int j = 0; j < nv; ++j) pos[j] = -1;
    for (int a = 0; a < n1; ++a) {
        if (keep[a] < 0 || keep[a] >= nv || (a > 0 && keep[a] <= keep[a - 1])) {
            free(pos); free(cnt); return -1;
        }
        pos[keep[a]] = a;
    }
    for (int j = 0; j < nv; ++j) {
        if (pos[j] >= 0) { assign[j] = pos[j]; continue; }
        int best = 0;
        double bc = cos_d(Ev + (size_t)j * d, Ev + (size_t)keep[0] * d, d);
        for (int a = 1; a < n1; ++a) {
            double c = cos_d(Ev + (size_t)j * d, Ev + (size_t)keep[a] * d, d);
            if (c > bc) { bc = c; best = a; }
        }
        assign[j] = best;
    }
    for (int a = 0; a < n1; ++a)
        for (int e = 0; e < d; ++e) merged[(size_t)a * d + e] = 0.0;
    for (int j = 0; j < nv; ++j) {
        int a = assign[j];
        cnt[a] += 1;
        for (int e = 0; e < d; ++e) merged[(size_t)a * d + e] += Ev[(size_t)j * d + e];
    }
    for (int a = 0; a < n1; ++a)
        for (int e = 0; e < d; ++e) merged[(size_t)a * d + e] /= (double)cnt[a];
    free(pos);
    free(cnt);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Sec. 4.4. One row of the attention map of query head h at absolute position
 * t: softmax over keys 0..t (causal, the query attends to itself) of
 * q_{t,h} . k_{k,g} / sqrt(dh), where g = h / (Hq / Hkv) is the key/value head
 * serving h. Q: [L, Hq, dh], K: [L, Hkv, dh]. prob: [t + 1].
 * ------------------------------------------------------------------------- */
static void po_attn_row(const double *Q, const double *K, int Hq, int Hkv, int dh, int h,
                        int t, double *prob) {
    int g = h / (Hq / Hkv);
    const double *q = Q + ((size_t)t * Hq + h) * dh;
    double scale = 1.0 / sqrt((double)dh);
    double mx = -INFINITY;
    for (int k = 0; k <= t; ++k) {
        prob[k] = dot_d(q, K + ((size_t)k * Hkv + g) * dh, dh) * scale;
        if (prob[k] > mx) mx = prob[k];
    }
    double z = 0.0;
    for (int k = 0; k <= t; ++k) z += exp(prob[k] - mx);
    for (int k = 0; k <= t; ++k) prob[k] = exp(prob[k] - mx) / z;
}

static int po_check_attn_args(int L, int Hq, int Hkv, int dh, const int *rows, int nr,
                              int vis_start, int nv) {
    if (L <= 0 || Hq <= 0 || Hkv <= 0 || dh <= 0 || Hq % Hkv != 0) return -1;
    if (nr <= 0 || !rows || nv <= 0 || vis_start < 0 || vis_start + nv > L) return -1;
    for (int a = 0; a < nr; ++a)
        if (rows[a] < 0 || rows[a] >= L) return -1;
    return 0;
}

/* ---------------------------------------------------------------------------
 * Sec. 4.4, S^vis and v:
 *   A_{h,j,i} = prob of text row rows[j] on visual column vis_start + i
 *               (0 when that column lies after the row, by causality)
 *   S_{j,i}   = (1/|heads|) sum_h A_{h,j,i}
 *   v_i       = (1/|rows|) sum_j S_{j,i}
 * heads: query-head ids; rows: absolute text positions. v: [nv].
 * ------------------------------------------------------------------------- */
int po_head_scores(const double *Q, const double *K, int L, int Hq, int Hkv, int dh,
                   const int *heads, int nh, const int *rows, int nr, int vis_start, int nv,
                   double *v) {
    if (po_check_attn_args(L, Hq, Hkv, dh, rows, nr, vis_start, nv) || !Q || !K || !v ||
        !heads || nh <= 0)
        return -1;
    for (int a = 0; a < nh; ++a)
        if (heads[a] < 0 || heads[a] >= Hq) return -1;
    double *prob = (double *)malloc(sizeof(double) * (size_t)L);
    double *S = (double *)malloc(sizeof(double) * (size_t)nv);
    if (!prob || !S) { free(prob); free(S); return -2; }
    for (int i = 0; i < nv; ++i) v[i] = 0.0;
    for (int j = 0; j < nr; ++j) {
        for (int i = 0; i < nv; ++i) S[i] = 0.0;
        for (int a = 0; a < nh; ++a) {
            po_attn_row(Q, K, Hq, Hkv, dh, heads[a], rows[j], prob);
            for (int i = 0; i < nv; ++i) {
                int col = vis_start + i;
                S[i] += (col <= rows[j]) ? prob[col] : 0.0;
            }
        }
        for (int i = 0; i < nv; ++i) v[i] += S[i] / (double)nh;
    }
    for (int i = 0; i < nv; ++i) v[i] /= (double)nr;
    free(prob);
    free(S);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Sec. 4.4, head confidence: C^h = sum over critical rows t of the population
 * variance (1/N) of A^cross_{h,t} over the nv visual columns. C: [Hq], every
 * query head.
 * ------------------------------------------------------------------------- */
int po_head_confidence(const double *Q, const double *K, int L, int Hq, int Hkv, int dh,
                       const int *rows, int nr, int vis_start, int nv, double *C) {
    if (po_check_attn_args(L, Hq, Hkv, dh, rows, nr, vis_start, nv) || !Q || !K || !C)
        return -1;
    double *prob = (double *)malloc(sizeof(double) * (size_t)L);
    if (!prob) return -2;
    for (int h = 0; h < Hq; ++h) {
        C[h] = 0.0;
        for (int j = 0; j < nr; ++j) {
            po_attn_row(Q, K, Hq, Hkv, dh, h, rows[j], prob);
            double mean = 0.0;
            for (int i = 0; i < nv; ++i) {
                int col = vis_start + i;
                mean += (col <= rows[j]) ? prob[col] : 0.0;
            }
            mean /= (double)nv;
            double var = 0.0;
            for (int i = 0; i < nv; ++i) {
                int col = vis_start + i;
                double a = ((col <= rows[j]) ? prob[col] : 0.0) - mean;
                var += a * a;
            }
            C[h] += var / (double)nv;
        }
    }
    free(prob);
    return 0;
}

/* ---------------------------------------------------------------------------
 * Rows that survive pruning, in order: the prefix rows [0, vis_start), the kept
 * visual rows vis_start + keep[a] (keep ascending), then every row after the
 * visual block up to seq_len. Writes src[0 .. out_len) and returns out_len
 * (= seq_len - nv + k), or -1 on an invalid argument.
 * ------------------------------------------------------------------------- */
int po_compact_map(int seq_len, int vis_start, int nv, const int *keep, int k, int *src) {
    if (vis_start < 0 || nv <= 0 || vis_start + nv > seq_len || k < 1 || k > nv || !keep ||
        !src)
        return -1;
    int o = 0;
    for (int r = 0; r < vis_start; ++r) src[o++] = r;
    for (int a = 0; a < k; ++a) {
        if (keep[a] < 0 || keep[a] >= nv || (a > 0 && keep[a] <= keep[a - 1])) return -1;
        src[o++] = vis_start + keep[a];
    }
    for (int r = vis_start + nv; r < seq_len; ++r) src[o++] = r;
    return o;
}

/* byte-exact gather of n rows of row_bytes each */
void po_gather_rows(const void *src, size_t row_bytes, const int *rows, int n, void *dst) {
    for (int o = 0; o < n; ++o)
        memcpy((char *)dst + (size_t)o * row_bytes,
               (const char *)src + (size_t)rows[o] * row_bytes, row_bytes);
}

/* ---------------------------------------------------------------------------
 * Sec. 4.4 end to end for a batch: scores, top-k, compaction. Used as the
 * timed CPU baseline. Per sample b (independent; OpenMP over samples):
 *   v     = po_head_scores(Q[b], K[b], rows = text_start[b] .. +text_len[b])
 *   keep  = po_topk(v, k)
 *   rows  = po_compact_map(seq_len[b], vis_start, nv, keep)
 *   hidden_out[b], K_out[b], V_out[b] = row gathers of the raw bytes;
 *   pos_out[p][b] = gather of pos[p][b] (np position rows)
 * Q, K are fp64 [B, Lmax, Hq|Hkv, dh]; hidden/Kraw/Vraw are raw bytes with
 * the given row sizes and Lmax rows per sample; pos int32 [np, B, Lmax].
 * Outputs: v_out [B, nv], idx_out [B, k], per-sample rows Lout = Lmax - nv + k.
 * threads <= 0 uses the OpenMP default.
 * ------------------------------------------------------------------------- */
int po_prune_batch(int B, int Lmax, const int *seq_len, const double *Q, const double *K,
                   int Hq, int Hkv, int dh, const int *heads, int nh, const int *text_start,
                   const int *text_len, int vis_start, int nv, int k, const void *hidden,
                   size_t hid_row_bytes, const void *Kraw, const void *Vraw,
                   size_t kv_row_bytes, const int32_t *pos, int np, double *v_out,
                   int *idx_out, void *hidden_out, void *K_out, void *V_out,
                   int32_t *pos_out, int *seq_len_out, int threads) {
    if (B <= 0 || Lmax <= 0 || k < 1 || k > nv) return -1;
    int Lout = Lmax - nv + k;
    int err = 0;
#ifdef _OPENMP
    if (threads > 0) omp_set_num_threads(threads);
#pragma omp parallel for schedule(dynamic, 1) reduction(| : err)
#endif
    for (int b = 0; b < B; ++b) {
        int nr = text_len[b];
        int *rows = (int *)malloc(sizeof(int) * (size_t)(nr > 0 ? nr : 1));
        int *src = (int *)malloc(sizeof(int) * (size_t)Lmax);
        if (!rows || !src) { free(rows); free(src); err |= 1; continue; }
        for (int j = 0; j < nr; ++j) rows[j] = text_start[b] + j;
        const double *Qb = Q + (size_t)b * Lmax * Hq * dh;
        const double *Kb = K + (size_t)b * Lmax * Hkv * dh;
        double *vb = v_out + (size_t)b * nv;
        int *ib = idx_out + (size_t)b * k;
        int e = po_head_scores(Qb, Kb, seq_len[b], Hq, Hkv, dh, heads, nh, rows, nr,
                               vis_start, nv, vb);
        if (!e) e = po_topk(vb, nv, k, ib);
        int n = e ? -1 : po_compact_map(seq_len[b], vis_start, nv, ib, k, src);
        if (n < 0) { err |= 1; free(rows); free(src); continue; }
        seq_len_out[b] = n;
        po_gather_rows((const char *)hidden + (size_t)b * Lmax * hid_row_bytes,
                       hid_row_bytes, src, n,
                       (char *)hidden_out + (size_t)b * Lout * hid_row_bytes);
        if (Kraw && K_out)
            po_gather_rows((const char *)Kraw + (size_t)b * Lmax * kv_row_bytes,
                           kv_row_bytes, src, n,
                           (char *)K_out + (size_t)b * Lout * kv_row_bytes);
        if (Vraw && V_out)
            po_gather_rows((const char *)Vraw + (size_t)b * Lmax * kv_row_bytes,
                           kv_row_bytes, src, n,
                           (char *)V_out + (size_t)b * Lout * kv_row_bytes);
        for (int p = 0; p < np; ++p)
            po_gather_rows(pos + ((size_t)p * B + b) * Lmax, sizeof(int32_t), src, n,
                           pos_out + ((size_t)p * B + b) * Lout);
        free(rows);
        free(src);
    }
    return err ? -1 : 0;
}

/* number of OpenMP threads a parallel region would use (1 without OpenMP) */
int po_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
