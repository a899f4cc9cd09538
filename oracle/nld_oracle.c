/*
 * nld_oracle.c -- plain, slow, fp64 CPU oracle for block attention over a
 * paged KV cache and for the two token-decision rules of tri-mode decoding.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may call, link or
 * load this file; only the tests, the smoke check and the bench's CPU
 * baseline do. It shares no code, header or table with the CUDA library.
 *
 * What it computes, by definition (each function cites its passage):
 *
 *  - Block attention (Sec. 2.2 attention pattern; Sec. 3 Mode 2 and Mode 3).
 *    A block of bl query tokens sits after a cached prefix of L_b tokens.
 *    Key t is visible to block row i when t < L_b (the clean prefix is fully
 *    visible), or t = L_b + j with j in J(i): J(i) = {0..bl-1} in the
 *    diffusion-draft pass (bidirectional inside the block) and {0..i} in the
 *    AR-verify pass (causal inside the block). Query head h reads KV head
 *    floor(h / G), G = Hq / Hkv. Logical key t lives in physical page
 *    page_table[b][t / P] at slot t mod P.
 *      s_t = scale * <q, k_t>,  m = max s_t,  w_t = exp(s_t - m),
 *      l = sum w_t,  o = sum w_t v_t / l,  lse = m + ln l.
 *  - Split-KV combine: partial results over disjoint key ranges merge as
 *      m* = max_s lse_s, c_s = exp(lse_s - m*), o = sum c_s o_s / sum c_s,
 *      lse = m* + ln sum c_s.
 *  - Acceptance (Sec. 3 Mode 3, linear self-speculation): the longest prefix
 *    of draft tokens equal to the verifier's predictions is accepted; the
 *    accepted length is the first mismatch index j*, or n if none.
 *  - Confidence-ranked unmasking (Sec. 3 Mode 2; Sec. 4 serial denoising
 *    commits the highest-confidence position): the k eligible positions with
 *    the largest confidence, ordered by (confidence descending, position
 *    ascending). -inf and NaN mark ineligible positions.
 *  - Threshold unmasking with a top-1 fallback (Sec. 2, confidence-based
 *    sampling) and greedy parallel acceptance against a serial target
 *    (Sec. 5, diffusion SOL construction): the positions one denoising step
 *    commits, in ascending order.
 *  - Logits -> (argmax id, max softmax probability) per position, the
 *    inputs of the two decisions (Sec. 2; Sec. 5).
 *  - Block KV commit into the paged slots after the prefix, with the prefix
 *    advanced by the committed rows (Sec. 3 Mode 3; Sec. 2 block refresh).
 *  - Block attention with a table mask over the block slots, and the
 *    structured mask of quadratic self-speculation (Sec. 3 variant; appendix
 *    Eq. quad_input) as one such table.
 *  - The AR-diffusion ensemble verifier: argmax and max of the mixture of
 *    the two predicted distributions (appendix, quadratic SS details).
 *
 * Build: gcc -O2 -fopenmp -ffp-contract=off -shared -fPIC (see build.py).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define NLDO_OK 0
#define NLDO_ERR_ARGS -1
#define NLDO_ERR_PAGE -2
#define NLDO_ERR_NOMEM -3

/* Exact widening of a bf16 bit pattern: the 16 bits are the top half of an
 * IEEE binary32, which converts to binary64 exactly. */
static double bf16_to_f64(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Mask of Sec. 2.2 / Sec. 3 for block row i (0-based) and logical key t.
 * Mode 2 takes the block part from a table: bit j of bm[i] makes block slot j
 * visible to row i (the structured mask of quadratic self-speculation,
 * Sec. 3 variant, is one such table). */
static int key_visible(long t, long L, int bl, int i, int mode, const uint32_t *bm)
{
    if (t < L) return 1;             /* clean prefix: always visible */
    long j = t - L;                  /* block slot of key t */
    if (j >= bl) return 0;           /* slots past the block hold nothing */
    if (mode == 0) return 1;         /* diffusion draft: bidirectional */
    if (mode == 2) return (int)((bm[i] >> j) & 1u);
    return j <= i;                   /* AR verify: causal, self included */
}

int nldo_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/*
 * One query row (b, i, h). Keys are restricted to the logical range
 * [key_begin, key_end) in addition to the mask (key_end < 0: no limit).
 * Writes o[D], *lse, and, when probs != NULL, probs[t] for t < L_b + bl
 * (0 for keys that are not used). A row with no usable key gets o = 0 and
 * lse = -inf.
 */
static int attn_row(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                    const int32_t *page_table, long L, int b, int i, int h,
                    int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                    int bl, int mode, const uint32_t *bm, double scale, long key_begin, long key_end,
                    double *s, char *use, double *o, double *lse, double *probs)
{
    const int G = Hq / Hkv;
    const int g = h / G;
    const long N = L + bl;
    const uint16_t *qrow = q + (((long)b * bl + i) * Hq + h) * (long)D;
    double m = -INFINITY;
    long nuse = 0;

    for (long t = 0; t < N; ++t) {
        use[t] = key_visible(t, L, bl, i, mode, bm) && t >= key_begin && (key_end < 0 || t < key_end);
        if (!use[t]) continue;
        long lp = t / P;
        if (lp >= max_pages) return NLDO_ERR_PAGE;
        int page = page_table[(long)b * max_pages + lp];
        if (page < 0 || page >= num_pages) return NLDO_ERR_PAGE;
        const uint16_t *krow = k + (((long)page * Hkv + g) * P + (t % P)) * (long)D;
        double dot = 0.0;
        for (int d = 0; d < D; ++d) dot += bf16_to_f64(qrow[d]) * bf16_to_f64(krow[d]);
        s[t] = scale * dot;
        if (s[t] > m) m = s[t];
        ++nuse;
    }
    for (int d = 0; d < D; ++d) o[d] = 0.0;
    if (nuse == 0) {
        *lse = -INFINITY;
        if (probs) for (long t = 0; t < N; ++t) probs[t] = 0.0;
        return NLDO_OK;
    }
    double l = 0.0;
    for (long t = 0; t < N; ++t) {
        if (!use[t]) continue;
        double w = exp(s[t] - m);
        l += w;
        int page = page_table[(long)b * max_pages + t / P];
        const uint16_t *vrow = v + (((long)page * Hkv + g) * P + (t % P)) * (long)D;
        for (int d = 0; d < D; ++d) o[d] += w * bf16_to_f64(vrow[d]);
    }
    for (int d = 0; d < D; ++d) o[d] /= l;
    *lse = m + log(l);
    if (probs)
        for (long t = 0; t < N; ++t) probs[t] = use[t] ? exp(s[t] - m) / l : 0.0;
    return NLDO_OK;
}

static int check_shape(int B, int Hq, int Hkv, int D, int P, int bl, int mode)
{
    if (B < 0 || Hq <= 0 || Hkv <= 0 || D <= 0 || P <= 0 || bl <= 0) return 0;
    if (Hq % Hkv != 0) return 0;
    if (mode != 0 && mode != 1 && !(mode == 2 && bl <= 32)) return 0;
    return 1;
}

/*
 * Block attention for every row. q [B, bl, Hq, D]; k, v [num_pages, Hkv, P, D]
 * (bf16 bits); page_table [B, max_pages]; prefix_lens [B].
 * out [B, bl, Hq, D], lse [B, Hq, bl] (fp64). probs: NULL, or
 * [B, Hq, bl, probs_stride] with probs_stride >= max_b (L_b + bl).
 */
static int block_attn_all(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                          const int32_t *page_table, const int32_t *prefix_lens,
                          int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                          int bl, int mode, const uint32_t *bm, double scale, long key_begin, long key_end,
                          double *out, double *lse, double *probs, long probs_stride)
{
    if (!check_shape(B, Hq, Hkv, D, P, bl, mode)) return NLDO_ERR_ARGS;
    if (mode == 2 && bm == NULL) return NLDO_ERR_ARGS;
    long maxN = 0;
    for (int b = 0; b < B; ++b) {
        if (prefix_lens[b] < 0) return NLDO_ERR_ARGS;
        if ((long)prefix_lens[b] + bl > maxN) maxN = (long)prefix_lens[b] + bl;
    }
    if (probs && probs_stride < maxN) return NLDO_ERR_ARGS;
    int status = NLDO_OK;
    long nrows = (long)B * Hq;
#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * (maxN > 0 ? maxN : 1));
        char *use = (char *)malloc(maxN > 0 ? maxN : 1);
        double *o = (double *)malloc(sizeof(double) * D);
        if (!s || !use || !o) {
#pragma omp atomic write
            status = NLDO_ERR_NOMEM;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (long bh = 0; bh < nrows; ++bh) {
                int b = (int)(bh / Hq), h = (int)(bh % Hq);
                for (int i = 0; i < bl; ++i) {
                    double l_out;
                    double *p = probs ? probs + ((bh * bl) + i) * probs_stride : NULL;
                    int rc = attn_row(q, k, v, page_table, prefix_lens[b], b, i, h, Hq, Hkv, D, P,
                                      num_pages, max_pages, bl, mode, bm, scale, key_begin, key_end,
                                      s, use, o, &l_out, p);
                    if (rc != NLDO_OK) {
#pragma omp atomic write
                        status = rc;
                        continue;
                    }
                    double *orow = out + (((long)b * bl + i) * Hq + h) * (long)D;
                    for (int d = 0; d < D; ++d) orow[d] = o[d];
                    lse[((long)b * Hq + h) * bl + i] = l_out;
                }
            }
        }
        free(s); free(use); free(o);
    }
    return status;
}

int nldo_block_attn(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                    const int32_t *page_table, const int32_t *prefix_lens,
                    int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                    int bl, int mode, double scale, long key_begin, long key_end,
                    double *out, double *lse, double *probs, long probs_stride)
{
    if (mode == 2) return NLDO_ERR_ARGS;  /* the table form has its own entry */
    return block_attn_all(q, k, v, page_table, prefix_lens, B, Hq, Hkv, D, P, num_pages, max_pages, bl,
                          mode, NULL, scale, key_begin, key_end, out, lse, probs, probs_stride);
}

/* Block attention whose block part follows a table: bit j of block_mask[i]
 * makes block slot j visible to block row i (bl <= 32); the prefix is
 * fully visible as in every mode. */
int nldo_block_attn_masked(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                           const int32_t *page_table, const int32_t *prefix_lens,
                           int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                           int bl, const uint32_t *block_mask, double scale,
                           double *out, double *lse, double *probs, long probs_stride)
{
    return block_attn_all(q, k, v, page_table, prefix_lens, B, Hq, Hkv, D, P, num_pages, max_pages, bl,
                          2, block_mask, scale, 0, -1, out, lse, probs, probs_stride);
}

/*
 * Block attention for selected rows only: rows[r] = (b, i, h) triples.
 * out [nrows, D], lse [nrows].
 */
int nldo_block_attn_rows(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                         const int32_t *page_table, const int32_t *prefix_lens,
                         int B, int Hq, int Hkv, int D, int P, int num_pages, int max_pages,
                         int bl, int mode, double scale, long nsel, const int32_t *rows,
                         double *out, double *lse)
{
    if (!check_shape(B, Hq, Hkv, D, P, bl, mode) || mode == 2) return NLDO_ERR_ARGS;
    long maxN = 0;
    for (int b = 0; b < B; ++b)
        if ((long)prefix_lens[b] + bl > maxN) maxN = (long)prefix_lens[b] + bl;
    int status = NLDO_OK;
#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * (maxN > 0 ? maxN : 1));
        char *use = (char *)malloc(maxN > 0 ? maxN : 1);
        if (!s || !use) {
#pragma omp atomic write
            status = NLDO_ERR_NOMEM;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (long r = 0; r < nsel; ++r) {
                int b = rows[3 * r], i = rows[3 * r + 1], h = rows[3 * r + 2];
                if (b < 0 || b >= B || i < 0 || i >= bl || h < 0 || h >= Hq) {
#pragma omp atomic write
                    status = NLDO_ERR_ARGS;
                    continue;
                }
                int rc = attn_row(q, k, v, page_table, prefix_lens[b], b, i, h, Hq, Hkv, D, P,
                                  num_pages, max_pages, bl, mode, NULL, scale, 0, -1,
                                  s, use, out + r * (long)D, lse + r, NULL);
                if (rc != NLDO_OK) {
#pragma omp atomic write
                    status = rc;
                }
            }
        }
        free(s); free(use);
    }
    return status;
}

/*
 * Split-KV combine. o_part [S, R, D], lse_part [S, R] -> out [R, D], lse [R].
 * Partials with lse = -inf carry no keys and get weight 0.
 */
void nldo_combine(const double *o_part, const double *lse_part, int S, long R, int D,
                  double *out, double *lse)
{
    for (long r = 0; r < R; ++r) {
        double m = -INFINITY;
        for (int s = 0; s < S; ++s)
            if (lse_part[(long)s * R + r] > m) m = lse_part[(long)s * R + r];
        double *orow = out + r * (long)D;
        for (int d = 0; d < D; ++d) orow[d] = 0.0;
        if (m == -INFINITY) { lse[r] = -INFINITY; continue; }
        double csum = 0.0;
        for (int s = 0; s < S; ++s) {
            double ls = lse_part[(long)s * R + r];
            if (ls == -INFINITY) continue;
            double c = exp(ls - m);
            csum += c;
            const double *op = o_part + ((long)s * R + r) * D;
            for (int d = 0; d < D; ++d) orow[d] += c * op[d];
        }
        for (int d = 0; d < D; ++d) orow[d] /= csum;
        lse[r] = m + log(csum);
    }
}

/* Longest accepted prefix: first j with draft[j] != verify[j], else n. */
void nldo_accept(const int32_t *draft, const int32_t *verify, int B, int n, int32_t *accepted)
{
    for (int b = 0; b < B; ++b) {
        int j = 0;
        while (j < n && draft[(long)b * n + j] == verify[(long)b * n + j]) ++j;
        accepted[b] = j;
    }
}

/* a ranks before b: larger confidence first; equal confidence -> lower index. */
static int ranks_before(float ca, int a, float cb, int b)
{
    if (ca > cb) return 1;
    if (ca < cb) return 0;
    return a < b;
}

/*
 * Top-k unmasking by confidence. conf [B, n] fp32. positions [B, k] in rank
 * order, -1 past the eligible count; num_selected [B] (nullable).
 * Eligible: not NaN and not -inf. Comparisons are made on the fp32 values
 * (+0 and -0 compare equal, so they tie and the lower index wins).
 */
void nldo_unmask(const float *conf, int B, int n, int k, int32_t *positions, int32_t *num_selected)
{
    int *idx = (int *)malloc(sizeof(int) * (n > 0 ? n : 1));
    for (int b = 0; b < B; ++b) {
        const float *c = conf + (long)b * n;
        int m = 0;
        for (int i = 0; i < n; ++i)
            if (!isnan(c[i]) && !(isinf(c[i]) && c[i] < 0)) idx[m++] = i;
        /* insertion sort: stable and obviously correct */
        for (int a = 1; a < m; ++a) {
            int x = idx[a], j = a - 1;
            while (j >= 0 && ranks_before(c[x], x, c[idx[j]], idx[j])) { idx[j + 1] = idx[j]; --j; }
            idx[j + 1] = x;
        }
        int sel = m < k ? m : k;
        for (int r = 0; r < k; ++r) positions[(long)b * k + r] = r < sel ? idx[r] : -1;
        if (num_selected) num_selected[b] = sel;
    }
    free(idx);
}

static int eligible(float c)
{
    return !isnan(c) && !(isinf(c) && c < 0);
}

/* Position of the highest eligible confidence (lower index on ties), or -1. */
static int top1(const float *c, int n)
{
    int best = -1;
    for (int i = 0; i < n; ++i)
        if (eligible(c[i]) && (best < 0 || ranks_before(c[i], i, c[best], best))) best = i;
    return best;
}

/*
 * Threshold unmasking (Sec. 2, confidence-based sampling: one denoising step
 * commits every masked position whose confidence exceeds the threshold),
 * with a top-1 fallback so that every step commits at least one position
 * while any is masked (the single highest-confidence position, as in the
 * fallback of Sec. 5 greedy acceptance). "Exceeds" is read as strictly
 * greater, compared in fp32. positions [B, n]: the committed positions in
 * ascending order, then -1; num_selected [B] (nullable). Eligible (still
 * masked): not NaN and not -inf.
 */
void nldo_unmask_threshold(const float *conf, int B, int n, float threshold, int32_t *positions,
                           int32_t *num_selected)
{
    for (int b = 0; b < B; ++b) {
        const float *c = conf + (long)b * n;
        int32_t *pos = positions + (long)b * n;
        int count = 0;
        for (int i = 0; i < n; ++i)
            if (eligible(c[i]) && c[i] > threshold) pos[count++] = i;
        if (count == 0) {
            const int best = top1(c, n);
            if (best >= 0) pos[count++] = best;
        }
        for (int r = count; r < n; ++r) pos[r] = -1;
        if (num_selected) num_selected[b] = count;
    }
}

/*
 * Greedy parallel acceptance (Sec. 5, diffusion SOL construction): one
 * iteration commits every masked position j whose argmax prediction equals
 * the serial target, {j : x_j = [M] and pred_j = target_j}; if there is none,
 * it commits the single highest-confidence masked position. pred, target
 * [B, n] int32; conf [B, n] fp32 marks the masked positions (eligible as
 * above) and ranks them for the fallback. Output as for
 * nldo_unmask_threshold.
 */
void nldo_greedy_accept(const int32_t *pred, const int32_t *target, const float *conf, int B, int n,
                        int32_t *positions, int32_t *num_selected)
{
    for (int b = 0; b < B; ++b) {
        const float *c = conf + (long)b * n;
        const int32_t *p = pred + (long)b * n;
        const int32_t *t = target + (long)b * n;
        int32_t *pos = positions + (long)b * n;
        int count = 0;
        for (int j = 0; j < n; ++j)
            if (eligible(c[j]) && p[j] == t[j]) pos[count++] = j;
        if (count == 0) {
            const int fallback = top1(c, n);
            if (fallback >= 0) pos[count++] = fallback;
        }
        for (int r = count; r < n; ++r) pos[r] = -1;
        if (num_selected) num_selected[b] = count;
    }
}

/*
 * Logits -> (argmax id, confidence) per position, the confidence being the
 * highest peak probability of the position's output distribution (Sec. 5,
 * serial denoising; Sec. 2, confidence-based sampling):
 *   m = max_v l_v over the non-NaN logits, id = the lowest v with l_v = m,
 *   conf = max_v softmax(l)_v = exp(m - lse) = 1 / sum_v exp(l_v - m).
 * logits bf16 bits [rows, ld] (the first `vocab` of each row are used).
 * A NaN logit never wins the argmax and makes the confidence NaN (the sum
 * takes it); a row with no logit above -inf gets id 0 and confidence 0.
 */
void nldo_logits_argmax(const uint16_t *logits, long rows, int vocab, long ld, int32_t *ids, double *conf)
{
    #pragma omp parallel for schedule(dynamic, 1)
    for (long r = 0; r < rows; ++r) {
        const uint16_t *row = logits + r * ld;
        double m = -INFINITY;
        int id = 0;
        for (int v = 0; v < vocab; ++v) {
            const double l = bf16_to_f64(row[v]);
            if (l > m) { m = l; id = v; }
        }
        ids[r] = id;
        if (m == -INFINITY) { conf[r] = 0.0; continue; }
        double sum = 0.0;
        for (int v = 0; v < vocab; ++v) sum += exp(bf16_to_f64(row[v]) - m);
        conf[r] = 1.0 / sum;
    }
}

/*
 * Block KV commit into the paged cache (Sec. 3 Mode 3: the accepted prefix is
 * committed to the verified prefix and the verifier's cache is rebuilt at the
 * rejection point; Sec. 2: a completed block's KV cache is refreshed). Row j
 * of the block (j < count_b; count_b = counts[b], or bl when counts is NULL)
 * is written to logical slot L_b + j, i.e. physical page
 * page_table[b][(L_b + j) / P], slot (L_b + j) mod P, for every KV head.
 * With `advance`, L_b becomes L_b + count_b afterwards (slots past it are
 * left as they are: they are simply no longer part of the prefix).
 * k_new, v_new bf16 bits [B, bl, Hkv, D]; pools [num_pages, Hkv, P, D].
 * A slot past the page table, or a page id outside the pool, is not written.
 */
void nldo_kv_commit(const uint16_t *k_new, const uint16_t *v_new, const int32_t *counts,
                    const int32_t *page_table, int32_t *prefix_lens, int advance,
                    uint16_t *k_pages, uint16_t *v_pages, int B, int Hkv, int D, int P,
                    int num_pages, int max_pages, int bl)
{
    for (int b = 0; b < B; ++b) {
        const long L = prefix_lens[b];
        const int count = counts ? counts[b] : bl;
        for (int j = 0; j < count; ++j) {
            const long t = L + j;
            if (t < 0 || t >= (long)max_pages * P) continue;
            const long page = page_table[(long)b * max_pages + t / P];
            if (page < 0 || page >= num_pages) continue;
            const long slot = t % P;
            for (int g = 0; g < Hkv; ++g) {
                const long src = (((long)b * bl + j) * Hkv + g) * D;
                const long dst = ((page * Hkv + g) * P + slot) * D;
                for (int d = 0; d < D; ++d) {
                    k_pages[dst + d] = k_new[src + d];
                    v_pages[dst + d] = v_new[src + d];
                }
            }
        }
        if (advance) prefix_lens[b] = (int32_t)(L + count);
    }
}

/*
 * The block layout and mask of quadratic self-speculation (Sec. 3 variant;
 * appendix, Eq. quad_input): after the verified prefix come the AR token
 * x_{n+1}, then k groups, each a speculative token x^t_{n+g+1} followed by k
 * fresh mask tokens: 1 + k + k^2 block slots. Reading of the structured
 * mask: the speculative chain (x_{n+1} and the k speculative tokens) is
 * causal among itself and sees no mask token, so its predictions verify the
 * previous drafts; the k masks of group g see the chain up to their own
 * speculative token and, bidirectionally, the masks of their group, so they
 * draft the next block for the case that verification accepts up to that
 * token. Writes masks[0 .. 1+k+k^2-1] (bit j: slot j visible); returns the
 * block length, or -1 when it exceeds 32 slots.
 */
int nldo_quadss_mask(int k, uint32_t *masks)
{
    const int n = 1 + k + k * k;
    if (k < 1 || n > 32) return -1;
    /* group of slot j: 0 for the AR token, g for the speculative token of
     * group g and for its masks; chain slots are the AR and speculative ones */
    int group[32], chain[32];
    group[0] = 0;
    chain[0] = 1;
    for (int g = 1; g <= k; ++g) {
        const int spec = 1 + (g - 1) * (k + 1);
        group[spec] = g;
        chain[spec] = 1;
        for (int r = 1; r <= k; ++r) {
            group[spec + r] = g;
            chain[spec + r] = 0;
        }
    }
    for (int i = 0; i < n; ++i) {
        uint32_t bits = 0;
        for (int j = 0; j < n; ++j) {
            int vis;
            if (chain[i])
                vis = chain[j] && j <= i;
            else
                vis = (chain[j] && group[j] <= group[i]) || (!chain[j] && group[j] == group[i]);
            if (vis) bits |= 1u << j;
        }
        masks[i] = bits;
    }
    return n;
}

/* softmax of one bf16 row into p[0..vocab) (fp64); all zero when no logit is above -inf */
static void softmax_row(const uint16_t *row, int vocab, double *p)
{
    double m = -INFINITY;
    for (int v = 0; v < vocab; ++v) {
        const double l = bf16_to_f64(row[v]);
        if (l > m) m = l;
    }
    if (m == -INFINITY) {
        for (int v = 0; v < vocab; ++v) p[v] = 0.0;
        return;
    }
    double sum = 0.0;
    for (int v = 0; v < vocab; ++v) sum += (p[v] = exp(bf16_to_f64(row[v]) - m));
    for (int v = 0; v < vocab; ++v) p[v] /= sum;
}

/*
 * AR-diffusion ensemble verifier (appendix, verification with the ensemble):
 * p_ens = lambda p_AR + (1 - lambda) p_diff over the vocabulary, from the
 * causal logits at a speculative token and the denoising logits at the mask
 * that follows it; ids = the lowest argmax of p_ens, conf = max p_ens.
 * A distribution with no logit above -inf contributes nothing. Logits are
 * finite or -inf. ar, diff bf16 bits [rows, ld].
 */
void nldo_ensemble_argmax(const uint16_t *ar, const uint16_t *diff, long rows, int vocab, long ld,
                          double lambda, int32_t *ids, double *conf)
{
    #pragma omp parallel
    {
        double *pa = (double *)malloc(sizeof(double) * (vocab > 0 ? vocab : 1));
        double *pb = (double *)malloc(sizeof(double) * (vocab > 0 ? vocab : 1));
        #pragma omp for schedule(dynamic, 1)
        for (long r = 0; r < rows; ++r) {
            softmax_row(ar + r * ld, vocab, pa);
            softmax_row(diff + r * ld, vocab, pb);
            double best = -1.0;
            int id = 0;
            for (int v = 0; v < vocab; ++v) {
                const double p = lambda * pa[v] + (1.0 - lambda) * pb[v];
                if (p > best) { best = p; id = v; }
            }
            ids[r] = id;
            conf[r] = best;
        }
        free(pa);
        free(pb);
    }
}
