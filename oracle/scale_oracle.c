/*
 * scale_oracle.c -- CPU fp64 oracle for the Similarity Chunk Rolling (SCR)
 * prefill path of SCALE (arXiv 2609.31568).
 *
 * TEST INFRASTRUCTURE. Only the test suite, the package smoke check and the
 * CPU-baseline leg of the benchmark load this library. The product path never
 * calls it, links it or reads anything it writes. It shares no code, header,
 * table or helper with the CUDA implementation.
 *
 * It takes the paper's steps in the paper's order and notation, in plain
 * double precision, one element at a time, with no blocking or fusion:
 *
 *   oracle_fingerprints       Eq. 6: v_i = mean of the multi-head queries of
 *                             sub-chunk X_i; ||v_i||_2 for the pre-normalised
 *                             v~_i = v_i / ||v_i|| of Sec. V-A1.
 *   oracle_anchor_clustering  Eq. 8 and Algorithm 1, run inside each outer
 *                             chunk (Sec. III-A, Algorithm 2 works per outer
 *                             chunk).
 *   oracle_block_reps         block representative key = mean of the block's
 *                             keys. The paper selects single tokens; this is
 *                             the block reading whose block size 1 case is the
 *                             paper's token rule exactly (see oracle_select).
 *   oracle_select             Eq. 9 with head soft-voting (Sec. V-A3,
 *                             "Selection function instantiation"): per-head
 *                             dot products of the anchor fingerprint with the
 *                             representatives, a softmax per head, a sum over
 *                             heads, top-k with ties to the lower index.
 *   oracle_attention_rows     Eq. 10 with the three key groups of Sec. V-A3
 *                             ("Sparse attention over the cluster"): sinks,
 *                             the selected blocks and the local window widened
 *                             to span the cluster, taken as a set, masked
 *                             causally (key at or before the query row).
 *
 * Readings of the paper where it is silent (each also listed in the design
 * notes of the repository):
 *   R1  block representative = mean of the block's post-RoPE keys;
 *   R2  selection logit z = sigma * v_a^(h) . r_b, sigma given (1 literally);
 *   R3  the per-head softmax runs over the candidate blocks only;
 *   R4  candidate blocks = blocks with at least one token in [n_sink, W_u),
 *       W_u = max(0, s_u - n_local); sinks and local window are not scored;
 *   R5  top-k ties go to the lower block index; output ascending;
 *   R6  query head h reads KV head floor(h / (H_q / H_kv));
 *   R7  local window of unit u = [W_u, e_u), clipped causally per row;
 *   R8  theta <= -1 admits every sub-chunk (fixed-size clusters);
 *   R9  a fingerprint of zero norm has cosine 0 with every other;
 *   R10 clusters never cross an outer-chunk boundary; the outer chunk length
 *       is a multiple of the sub-chunk length.
 *
 * Inputs are bf16 bit patterns (uint16), widened exactly to double.
 * Return value: 0 on success, -1 on an invalid argument.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_to_f64(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ---------------------------------------------------------------------------
 * Eq. 6: v_i = (1/|X_i|) sum_{t in X_i} q_{i,t}, with q_{i,t} the multi-head
 * query of token t (all H_q heads concatenated, d = H_q * d_h). Sub-chunk i
 * covers tokens [i L, min(N, (i+1) L)) (Sec. III-A; the last one may be
 * shorter). Also writes ||v_i||_2 (Sec. V-A1).
 *   q      [N][Hq][dh] bf16
 *   v      [M][Hq*dh]  out, M = ceil(N / L)
 *   norms  [M]         out
 * ------------------------------------------------------------------------- */
int oracle_fingerprints(const uint16_t *q, int64_t N, int Hq, int dh, int L,
                        double *v, double *norms)
{
    if (!q || !v || !norms || N <= 0 || Hq <= 0 || dh <= 0 || L <= 0) return -1;
    const int64_t D = (int64_t)Hq * dh;
    const int64_t M = (N + L - 1) / L;
    for (int64_t i = 0; i < M; ++i) {
        const int64_t t0 = i * L;
        const int64_t t1 = (t0 + L < N) ? t0 + L : N;
        double *vi = v + i * D;
        for (int64_t c = 0; c < D; ++c) vi[c] = 0.0;
        for (int64_t t = t0; t < t1; ++t)
            for (int64_t c = 0; c < D; ++c) vi[c] += bf16_to_f64(q[t * D + c]);
        double ss = 0.0;
        for (int64_t c = 0; c < D; ++c) {
            vi[c] /= (double)(t1 - t0);
            ss += vi[c] * vi[c];
        }
        norms[i] = sqrt(ss);
    }
    return 0;
}

/* cos(v_a, v_j) as the dot product of the pre-normalised v~ (Sec. V-A1). */
static double cosine(const double *v, const double *norms, int64_t D, int64_t a, int64_t j)
{
    if (norms[a] == 0.0 || norms[j] == 0.0) return 0.0; /* R9 */
    double s = 0.0;
    for (int64_t c = 0; c < D; ++c)
        s += (v[a * D + c] / norms[a]) * (v[j * D + c] / norms[j]);
    return s;
}

/* ---------------------------------------------------------------------------
 * Algorithm 1 (anchor-based clustering), admission rule Eq. 8, applied to the
 * sub-chunks of each outer chunk separately (Algorithm 2 runs per outer chunk;
 * R10). Cluster size cap: |C_a| * L < L_max with L_max = S_max * L, i.e.
 * |C_a| < S_max.
 *   v, norms        from oracle_fingerprints, M sub-chunks of dimension D
 *   S_max           L_max / L
 *   per_outer       sub-chunks per outer chunk (L_outer / L)
 *   unit_start      [M+1] out: cluster u = sub-chunks [unit_start[u], unit_start[u+1])
 *   n_units         out: |P| summed over outer chunks
 *   margin          out: min |cos - theta| over the comparisons that decided an
 *                   admission (+inf when none did), to flag near-threshold cases
 * ------------------------------------------------------------------------- */
int oracle_anchor_clustering(const double *v, const double *norms, int64_t M, int64_t D,
                             int S_max, int64_t per_outer, double theta,
                             int32_t *unit_start, int32_t *n_units, double *margin)
{
    if (!v || !norms || !unit_start || !n_units || M <= 0 || D <= 0 || S_max <= 0 || per_outer <= 0)
        return -1;
    const int always = theta <= -1.0; /* R8 */
    int32_t P = 0;
    double mg = INFINITY;
    for (int64_t c0 = 0; c0 < M; c0 += per_outer) {
        const int64_t c1 = (c0 + per_outer < M) ? c0 + per_outer : M;
        int64_t a = c0;
        while (a < c1) {
            unit_start[P++] = (int32_t)a;
            int64_t size = 1;
            int64_t j = a + 1;
            while (j < c1 && size < S_max) {
                int admit = 1;
                if (!always) {
                    double cs = cosine(v, norms, D, a, j);
                    if (fabs(cs - theta) < mg) mg = fabs(cs - theta);
                    admit = cs >= theta;
                }
                if (!admit) break;
                ++size;
                ++j;
            }
            a = j;
        }
    }
    unit_start[P] = (int32_t)M;
    *n_units = P;
    *margin = mg;
    return 0;
}

/* ---------------------------------------------------------------------------
 * Block representative keys (R1): r_b^(j) = mean of K_t^(j) over the tokens t
 * of block b = [b B, min(N, (b+1) B)).
 *   k     [N][Hkv][dh] bf16
 *   reps  [Hkv][nb][dh] out, nb = ceil(N / B)
 * ------------------------------------------------------------------------- */
int oracle_block_reps(const uint16_t *k, int64_t N, int Hkv, int dh, int B, double *reps)
{
    if (!k || !reps || N <= 0 || Hkv <= 0 || dh <= 0 || B <= 0) return -1;
    const int64_t nb = (N + B - 1) / B;
    for (int j = 0; j < Hkv; ++j)
        for (int64_t b = 0; b < nb; ++b) {
            const int64_t t0 = b * B;
            const int64_t t1 = (t0 + B < N) ? t0 + B : N;
            double *r = reps + ((int64_t)j * nb + b) * dh;
            for (int d = 0; d < dh; ++d) {
                double s = 0.0;
                for (int64_t t = t0; t < t1; ++t)
                    s += bf16_to_f64(k[(t * Hkv + j) * dh + d]);
                r[d] = s / (double)(t1 - t0);
            }
        }
    return 0;
}

/* Unit u's first sub-chunk (the anchor a) and token range [s_u, e_u). */
static void unit_range(int per_subchunk, const int32_t *unit_start, int64_t u, int64_t L, int64_t N,
                       int64_t *anchor, int64_t *s, int64_t *e)
{
    int64_t a, b;
    if (per_subchunk) {
        a = u;
        b = u + 1;
    } else {
        a = unit_start[u];
        b = unit_start[u + 1];
    }
    *anchor = a;
    *s = a * L;
    *e = (b * L < N) ? b * L : N;
}

typedef struct {
    double score;
    int32_t b;
} scored_t;

/* Descending score, then ascending block index (R5). */
static int cmp_scored(const void *x, const void *y)
{
    const scored_t *p = (const scored_t *)x, *q = (const scored_t *)y;
    if (p->score > q->score) return -1;
    if (p->score < q->score) return 1;
    return (p->b > q->b) - (p->b < q->b);
}

static int cmp_i32(const void *x, const void *y)
{
    int32_t p = *(const int32_t *)x, q = *(const int32_t *)y;
    return (p > q) - (p < q);
}

/* ---------------------------------------------------------------------------
 * Cluster-level selection, Eq. 9: I_C = S(v_a, K_cache), with S the head
 * soft-voting rule (Sec. V-A3): for each query head h, logits
 * z_{h,b} = sigma * v_a^(h) . r_b^(floor(h/g)) over the candidate blocks (R2,
 * R3, R4, R6), p_h = softmax_b(z_h), score_b = sum_h p_{h,b}; the k blocks of
 * highest score (ties to the lower index, R5), listed in ascending order.
 * Baseline mode (per_subchunk != 0) makes every sub-chunk its own unit, the
 * per-sub-chunk retrieval of Sec. III-A.
 *   reps        [Hkv][nb][dh] from oracle_block_reps
 *   v           [M][Hq*dh] from oracle_fingerprints (raw v_a, not v~, Sec. V-A3)
 *   unit_start  [n_units+1] (ignored in baseline mode, where n_units = M)
 *   sel         [n_units][k] out, ascending, -1 padded
 *   sel_count   [n_units] out: min(k, |Cand(u)|)
 *   cand_count  [n_units] out: |Cand(u)| (a retrieval call happens iff > 0)
 *   gap         [n_units] out: (s_k - s_{k+1}) / s_k when |Cand| > k, else +inf
 *   scores      [n_units][nb] out (nullable): score_b on Cand(u), NaN elsewhere
 * ------------------------------------------------------------------------- */
int oracle_select(int Hq, int Hkv, int dh, int64_t N, int L, int B, int k, int n_sink, int n_local,
                  double sigma, int per_subchunk, const double *reps, const double *v,
                  const int32_t *unit_start, int64_t n_units, int32_t *sel, int32_t *sel_count,
                  int32_t *cand_count, double *gap, double *scores)
{
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv || dh <= 0 || N <= 0 || L <= 0 || B <= 0 || k < 0 ||
        n_sink < 0 || n_local < 0 || !reps || !v || (!per_subchunk && !unit_start) || !sel ||
        !sel_count || !cand_count || !gap)
        return -1;
    const int g = Hq / Hkv;
    const int64_t nb = (N + B - 1) / B;
    const int64_t D = (int64_t)Hq * dh;
    int err = 0;
    /* Units are independent; each thread takes whole units with its own
     * scratch, so the arithmetic of a unit is the same as in a serial loop. */
#pragma omp parallel
    {
        scored_t *cand = (scored_t *)malloc(sizeof(scored_t) * (size_t)nb);
        double *z = (double *)malloc(sizeof(double) * (size_t)nb);
        double *score = (double *)malloc(sizeof(double) * (size_t)nb);
        const int ok = cand && z && score;
        if (!ok) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int64_t u = 0; u < n_units; ++u) {
            if (!ok) continue;
            int64_t a, s, e;
            unit_range(per_subchunk, unit_start, u, L, N, &a, &s, &e);
            const int64_t W = (s - n_local > 0) ? s - n_local : 0;

            /* R4: candidate blocks have a token in [n_sink, W). */
            int64_t nc = 0;
            for (int64_t b = 0; b < nb; ++b) {
                score[b] = NAN;
                if (b * B < W && (b + 1) * B > n_sink) cand[nc++].b = (int32_t)b;
            }
            for (int64_t i = 0; i < nc; ++i) score[cand[i].b] = 0.0;

            for (int h = 0; h < Hq && nc > 0; ++h) {
                const double *vh = v + a * D + (int64_t)h * dh;
                const double *rj = reps + (int64_t)(h / g) * nb * dh;
                double zmax = -INFINITY;
                for (int64_t i = 0; i < nc; ++i) {
                    const double *r = rj + (int64_t)cand[i].b * dh;
                    double dot = 0.0;
                    for (int d = 0; d < dh; ++d) dot += vh[d] * r[d];
                    z[i] = sigma * dot;
                    if (z[i] > zmax) zmax = z[i];
                }
                double den = 0.0;
                for (int64_t i = 0; i < nc; ++i) den += exp(z[i] - zmax);
                for (int64_t i = 0; i < nc; ++i) score[cand[i].b] += exp(z[i] - zmax) / den;
            }

            for (int64_t i = 0; i < nc; ++i) cand[i].score = score[cand[i].b];
            qsort(cand, (size_t)nc, sizeof(scored_t), cmp_scored);
            const int64_t take = nc < k ? nc : k;
            int32_t *su = sel + u * (int64_t)k;
            for (int64_t i = 0; i < k; ++i) su[i] = -1;
            for (int64_t i = 0; i < take; ++i) su[i] = cand[i].b;
            qsort(su, (size_t)take, sizeof(int32_t), cmp_i32);
            sel_count[u] = (int32_t)take;
            cand_count[u] = (int32_t)nc;
            gap[u] = (nc > k && k > 0) ? (cand[k - 1].score - cand[k].score) / cand[k - 1].score : INFINITY;
            if (scores)
                for (int64_t b = 0; b < nb; ++b) scores[u * nb + b] = score[b];
        }
        free(cand); free(z); free(score);
    }
    return err ? -1 : 0;
}

/* ---------------------------------------------------------------------------
 * Sparse attention, Eq. 10, for the query rows listed in `rows` (token
 * positions). Row p lies in unit u = [s_u, e_u). Its key set is
 *   K(p) = ( [0, n_sink) U (union of selected blocks of u) U [W_u, e_u) ) n [0, p]
 * taken as a set (Sec. V-A3: the three groups are de-duplicated; the causal
 * mask keeps keys at or before the row). For each head h:
 *   o = sum_{t in K(p)} softmax_t( attn_scale * q_p^(h) . k_t^(floor(h/g)) ) v_t^(floor(h/g)).
 *   q       [N][Hq][dh] bf16;  k, v  [N][Hkv][dh] bf16
 *   sel     [n_units][k], sel_count [n_units] (the selection to attend with)
 *   out     [n_rows][Hq][dh] out
 * ------------------------------------------------------------------------- */
int oracle_attention_rows(int Hq, int Hkv, int dh, int64_t N, int L, int B, int k, int n_sink,
                          int n_local, double attn_scale, int per_subchunk, const uint16_t *q,
                          const uint16_t *kc, const uint16_t *vc, const int32_t *unit_start,
                          int64_t n_units, const int32_t *sel, const int32_t *sel_count,
                          const int64_t *rows, int64_t n_rows, double *out)
{
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv || dh <= 0 || N <= 0 || L <= 0 || B <= 0 || k < 0 ||
        n_sink < 0 || n_local < 0 || !q || !kc || !vc || (!per_subchunk && !unit_start) ||
        (k > 0 && !sel) || !sel_count || !rows || !out)
        return -1;
    for (int64_t r = 0; r < n_rows; ++r)
        if (rows[r] < 0 || rows[r] >= N) return -1;
    const int g = Hq / Hkv;
    const int64_t nb = (N + B - 1) / B;
    int bad = 0;

#pragma omp parallel
    {
        double *logit = (double *)malloc(sizeof(double) * (size_t)N);
        int64_t *keys = (int64_t *)malloc(sizeof(int64_t) * (size_t)N);
        unsigned char *chosen = (unsigned char *)malloc((size_t)nb);
        if (!logit || !keys || !chosen) {
#pragma omp atomic write
            bad = 1;
        }
#pragma omp for schedule(dynamic, 4)
        for (int64_t r = 0; r < n_rows; ++r) {
            if (!logit || !keys || !chosen) continue;
            const int64_t p = rows[r];
            /* The unit containing p. */
            int64_t u = -1, a = 0, s = 0, e = 0;
            for (int64_t uu = 0; uu < n_units; ++uu) {
                unit_range(per_subchunk, unit_start, uu, L, N, &a, &s, &e);
                if (s <= p && p < e) { u = uu; break; }
            }
            if (u < 0) {
#pragma omp atomic write
                bad = 1;
                continue;
            }
            const int64_t W = (s - n_local > 0) ? s - n_local : 0;
            memset(chosen, 0, (size_t)nb);
            for (int32_t i = 0; i < sel_count[u]; ++i) {
                const int32_t b = sel[u * (int64_t)k + i];
                if (b >= 0 && b < nb) chosen[b] = 1;
            }
            int64_t nk = 0;
            for (int64_t t = 0; t <= p; ++t)
                if (t < n_sink || chosen[t / B] || t >= W) keys[nk++] = t;

            for (int h = 0; h < Hq; ++h) {
                const int j = h / g;
                const uint16_t *qh = q + (p * Hq + h) * (int64_t)dh;
                double m = -INFINITY;
                for (int64_t i = 0; i < nk; ++i) {
                    const uint16_t *kt = kc + (keys[i] * Hkv + j) * (int64_t)dh;
                    double dot = 0.0;
                    for (int d = 0; d < dh; ++d) dot += bf16_to_f64(qh[d]) * bf16_to_f64(kt[d]);
                    logit[i] = attn_scale * dot;
                    if (logit[i] > m) m = logit[i];
                }
                double den = 0.0;
                for (int64_t i = 0; i < nk; ++i) {
                    logit[i] = exp(logit[i] - m);
                    den += logit[i];
                }
                double *o = out + (r * Hq + h) * (int64_t)dh;
                for (int d = 0; d < dh; ++d) o[d] = 0.0;
                for (int64_t i = 0; i < nk; ++i) {
                    const uint16_t *vt = vc + (keys[i] * Hkv + j) * (int64_t)dh;
                    const double w = logit[i] / den;
                    for (int d = 0; d < dh; ++d) o[d] += w * bf16_to_f64(vt[d]);
                }
            }
        }
        free(logit);
        free(keys);
        free(chosen);
    }
    return bad ? -1 : 0;
}
