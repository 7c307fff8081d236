/*
 * specflash_oracle.c -- plain, slow, fp64 CPU oracle for the SpecFLASH
 * target-model verification step (arXiv 2505.12728).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the correctness reference that the
 * CUDA path is compared against.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load it.  The product library never
 * links, loads or calls it, and it shares no code, header, table or helper
 * with the CUDA path.
 *
 * What it computes (all arithmetic in double precision):
 *
 *   1. Verification attention (Sec. 3.1, "Preliminaries": the target model
 *      scores the K candidate tokens in parallel in a single forward pass
 *      against its cache of visual-then-text tokens).  For every sequence b,
 *      new query row i < n_q and query head h, with KV head h / (H_q / H_kv):
 *      the visible keys are the L_b prefix tokens plus draft rows 0..i
 *      (causal inside the draft block), s_t = scale * <q, k_t>,
 *      lse = log sum_t exp(s_t), o = sum_t exp(s_t - lse) v_t.
 *      This is the plain definition; no blocking, no online softmax.
 *
 *   2. Decode attention: one query against T contiguous keys.  A separate,
 *      independently written routine, so that "a k-row verify equals k
 *      sequential decodes" (the K = 1 degenerate case of the ablation on the
 *      draft length K) can be checked.
 *
 *   3. Acceptance (Sec. 3.1 and Sec. 3.3, the token-wise acceptance-rejection
 *      rule of the speculative-sampling method the paper cites): per sequence,
 *      candidate T'_{i+1} is accepted with probability min(1, p_i(x)/q_i(x)),
 *      the candidates are examined in order up to the first rejection j, and
 *      the token at position j is drawn from the residual distribution
 *      norm(max(0, p_j - q_j)), or from the bonus row p_k when all K drafts
 *      were accepted.  At temperature 0 (greedy decoding, Sec. 4.2) a draft is
 *      accepted iff it equals the argmax of the target logits.
 *
 *   4. KV commit after acceptance, draft-tail sampling (Algorithm 1) and
 *      visual token compression (Sec. 3.2, Eq. 3), each described at its
 *      function below.
 *
 * Readings of points the paper leaves open (each one is listed with its
 * reason in the design notes of the repository):
 *   - acceptance test: u * q(x) < p(x) with a strict "<" (u in [0,1));
 *   - greedy argmax ties go to the lowest token id; the argmax is taken on
 *     the raw fp32 logits;
 *   - all K accepted: a bonus token is drawn from row K of the target logits;
 *   - uniforms: u_0..u_{K-1} for the K tests, u_K for the single final draw;
 *   - residual with zero mass (rounding only): draw from p_j instead;
 *   - inverse CDF in ascending token id: the smallest x with u*S < C(x); if
 *     rounding leaves none, the last x with non-zero mass;
 *   - temperature: p = softmax(logits / tau); q is used as given;
 *   - scores are scaled by `scale` (1/sqrt(d) unless given); the LSE is the
 *     natural log of the sum of exp of the scaled scores.
 *
 * Every function here is pinned by the not-gpu tests against closed forms,
 * library routines, brute force and the distributional guarantee of the
 * acceptance rule; none is "parity unpinned".
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG 1
#define ORACLE_ERR_BAD_PAGE 2
#define ORACLE_ERR_BAD_TOKEN 3
#define ORACLE_ERR_NOMEM 4

/* bf16 is the upper half of an IEEE binary32; widening is exact. */
static double oracle_bf16_value(uint16_t bits)
{
    uint32_t w = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------------ */
/* Decode attention: one query row q[d] against keys k[T][d], values v[T][d]. */
/* ------------------------------------------------------------------------ */
int oracle_decode_attention(const double *q, const double *k, const double *v,
                            int T, int d, double scale, double *o,
                            double *lse_out)
{
    if (T <= 0 || d <= 0 || !q || !k || !v || !o)
        return ORACLE_ERR_ARG;
    double *s = (double *)malloc(sizeof(double) * (size_t)T);
    if (!s)
        return ORACLE_ERR_NOMEM;

    double smax = -INFINITY;
    for (int t = 0; t < T; ++t) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c)
            acc += q[c] * k[(size_t)t * d + c];
        s[t] = scale * acc;
        if (s[t] > smax)
            smax = s[t];
    }
    double z = 0.0;
    for (int t = 0; t < T; ++t)
        z += exp(s[t] - smax);
    double lse = smax + log(z);

    for (int c = 0; c < d; ++c)
        o[c] = 0.0;
    for (int t = 0; t < T; ++t) {
        double w = exp(s[t] - lse);
        for (int c = 0; c < d; ++c)
            o[c] += w * v[(size_t)t * d + c];
    }
    if (lse_out)
        *lse_out = lse;
    free(s);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------ */
/* Verification attention over a paged cache.                               */
/*                                                                          */
/* q        bf16 bits [B][n_q][H_q][d]                                      */
/* k_cache  bf16 bits [num_pages][H_kv][page_size][d]   (v_cache the same)  */
/* block_table [B][max_pages_per_seq]: logical page -> physical page        */
/* seq_lens [B]: L_b + n_q (the draft rows' K/V are already in the cache)   */
/* out [B][n_q][H_q][d], lse [B][n_q][H_q] (lse may be NULL)                */
/*                                                                          */
/* Only the rows selected by (b_sel, i_sel, h_sel) are computed when those   */
/* are >= 0 (a negative selector means "all"), so that full-size workloads  */
/* can be checked on sampled rows.                                          */
/* ------------------------------------------------------------------------ */
static int oracle_verify_one_row(const uint16_t *q, const uint16_t *k_cache,
                                 const uint16_t *v_cache,
                                 const int32_t *block_table,
                                 const int32_t *seq_lens, int b, int i, int h,
                                 int n_q, int H_q, int H_kv, int d,
                                 int page_size, int num_pages,
                                 int max_pages_per_seq, double scale,
                                 double *out, double *lse)
{
    const int group = H_q / H_kv;
    const int h_kv = h / group;
    const int T = seq_lens[b];
    const int L = T - n_q;          /* prefix length before the draft block */
    const int visible = L + i + 1;  /* prefix + draft rows 0..i            */

    const uint16_t *qrow = q + (((size_t)b * n_q + i) * H_q + h) * d;
    double *s = (double *)malloc(sizeof(double) * (size_t)visible);
    if (!s)
        return ORACLE_ERR_NOMEM;

    /* scores */
    double smax = -INFINITY;
    for (int t = 0; t < visible; ++t) {
        int logical_page = t / page_size;
        int slot = t % page_size;
        int page = block_table[(size_t)b * max_pages_per_seq + logical_page];
        if (page < 0 || page >= num_pages) {
            free(s);
            return ORACLE_ERR_BAD_PAGE;
        }
        const uint16_t *krow =
            k_cache + (((size_t)page * H_kv + h_kv) * page_size + slot) * d;
        double acc = 0.0;
        for (int c = 0; c < d; ++c)
            acc += oracle_bf16_value(qrow[c]) * oracle_bf16_value(krow[c]);
        s[t] = scale * acc;
        if (s[t] > smax)
            smax = s[t];
    }
    double z = 0.0;
    for (int t = 0; t < visible; ++t)
        z += exp(s[t] - smax);
    const double row_lse = smax + log(z);

    double *orow = out + (((size_t)b * n_q + i) * H_q + h) * d;
    for (int c = 0; c < d; ++c)
        orow[c] = 0.0;
    for (int t = 0; t < visible; ++t) {
        int page = block_table[(size_t)b * max_pages_per_seq + t / page_size];
        const uint16_t *vrow =
            v_cache +
            (((size_t)page * H_kv + h_kv) * page_size + (t % page_size)) * d;
        double w = exp(s[t] - row_lse);
        for (int c = 0; c < d; ++c)
            orow[c] += w * oracle_bf16_value(vrow[c]);
    }
    if (lse)
        lse[((size_t)b * n_q + i) * H_q + h] = row_lse;
    free(s);
    return ORACLE_OK;
}

int oracle_verify_attention(const uint16_t *q, const uint16_t *k_cache,
                            const uint16_t *v_cache, const int32_t *block_table,
                            const int32_t *seq_lens, int B, int n_q, int H_q,
                            int H_kv, int d, int page_size, int num_pages,
                            int max_pages_per_seq, double scale, int b_sel,
                            int i_sel, int h_sel, double *out, double *lse)
{
    if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !out)
        return ORACLE_ERR_ARG;
    if (B <= 0 || n_q <= 0 || H_q <= 0 || H_kv <= 0 || d <= 0 ||
        page_size <= 0 || num_pages <= 0 || max_pages_per_seq <= 0)
        return ORACLE_ERR_ARG;
    if (H_q % H_kv != 0)
        return ORACLE_ERR_ARG;
    for (int b = 0; b < B; ++b) {
        if (seq_lens[b] < n_q ||
            seq_lens[b] > (long long)max_pages_per_seq * page_size)
            return ORACLE_ERR_ARG;
    }
    if (scale == 0.0)
        scale = 1.0 / sqrt((double)d);

    int status = ORACLE_OK;
    const long long rows = (long long)B * n_q * H_q;
#pragma omp parallel for schedule(dynamic, 1)
    for (long long r = 0; r < rows; ++r) {
        int h = (int)(r % H_q);
        int i = (int)((r / H_q) % n_q);
        int b = (int)(r / ((long long)H_q * n_q));
        if ((b_sel >= 0 && b != b_sel) || (i_sel >= 0 && i != i_sel) ||
            (h_sel >= 0 && h != h_sel))
            continue;
        int st = oracle_verify_one_row(q, k_cache, v_cache, block_table,
                                       seq_lens, b, i, h, n_q, H_q, H_kv, d,
                                       page_size, num_pages, max_pages_per_seq,
                                       scale, out, lse);
        if (st != ORACLE_OK) {
#pragma omp critical
            status = st;
        }
    }
    return status;
}

/* ------------------------------------------------------------------------ */
/* Target distribution of one verified position: p = softmax(logits / tau).  */
/* ------------------------------------------------------------------------ */
int oracle_target_probs(const float *logits, int V, double tau, double *p)
{
    if (!logits || !p || V <= 0 || !(tau > 0.0))
        return ORACLE_ERR_ARG;
    double zmax = -INFINITY;
    for (int x = 0; x < V; ++x) {
        double z = (double)logits[x] / tau;
        if (z > zmax)
            zmax = z;
    }
    double sum = 0.0;
    for (int x = 0; x < V; ++x) {
        p[x] = exp((double)logits[x] / tau - zmax);
        sum += p[x];
    }
    for (int x = 0; x < V; ++x)
        p[x] /= sum;
    return ORACLE_OK;
}

/* Greedy decoding's choice: the first index holding the largest logit. */
int oracle_argmax(const float *logits, int V)
{
    int best = 0;
    for (int x = 1; x < V; ++x)
        if (logits[x] > logits[best])
            best = x;
    return best;
}

/* ------------------------------------------------------------------------ */
/* Acceptance for a batch of sequences.                                     */
/*                                                                          */
/* target_logits [B][k+1][V] fp32: row i scores draft i, row k is the bonus */
/* draft_probs   [B][k][V]   fp32: q_i, used as given                        */
/* draft_tokens  [B][k]      int32: T'_1..T'_k                              */
/* uniforms      [B][k+1]    fp32 in [0,1)                                  */
/* temperature   [B]         fp32: <= 0 means greedy for that sequence       */
/* outputs: num_accepted [B]; out_tokens [B][k+1] (first num_accepted + 1    */
/* valid, the rest -1); accept_ratio [B][k] = min(1, p/q) (greedy: 1 or 0),  */
/* may be NULL; margin [B][k+1] (may be NULL): for each test actually       */
/* evaluated |u_i - p/q| (q = 0: +inf), for the final draw the distance of  */
/* u_k to the nearest normalised CDF boundary; +inf where no floating-point */
/* comparison decides the outcome.                                          */
/* ------------------------------------------------------------------------ */
int oracle_accept(const float *target_logits, const float *draft_probs,
                  const int32_t *draft_tokens, const float *uniforms,
                  const float *temperature, int B, int k, int V,
                  int32_t *num_accepted, int32_t *out_tokens,
                  double *accept_ratio, double *margin)
{
    if (!target_logits || !draft_probs || !draft_tokens || !uniforms ||
        !temperature || !num_accepted || !out_tokens)
        return ORACLE_ERR_ARG;
    if (B <= 0 || k <= 0 || V <= 0)
        return ORACLE_ERR_ARG;
    for (long long n = 0; n < (long long)B * k; ++n)
        if (draft_tokens[n] < 0 || draft_tokens[n] >= V)
            return ORACLE_ERR_BAD_TOKEN;

    double *p = (double *)malloc(sizeof(double) * (size_t)V);
    double *r = (double *)malloc(sizeof(double) * (size_t)V);
    if (!p || !r) {
        free(p);
        free(r);
        return ORACLE_ERR_NOMEM;
    }

    for (int b = 0; b < B; ++b) {
        const float tau = temperature[b];
        const int greedy = !(tau > 0.0f);
        const float *rows = target_logits + (size_t)b * (k + 1) * V;
        const float *qrows = draft_probs + (size_t)b * k * V;
        const int32_t *x = draft_tokens + (size_t)b * k;
        const float *u = uniforms + (size_t)b * (k + 1);
        double *mg = margin ? margin + (size_t)b * (k + 1) : NULL;
        if (mg)
            for (int i = 0; i <= k; ++i)
                mg[i] = INFINITY;

        /* Score every draft (the target computes all rows in one pass), and
         * take the decisions in order up to the first rejection j. */
        int j = k;
        for (int i = 0; i < k; ++i) {
            const float *row = rows + (size_t)i * V;
            int accept;
            double ratio;
            double m = INFINITY;
            if (greedy) {
                accept = (x[i] == oracle_argmax(row, V));
                ratio = accept ? 1.0 : 0.0;
            } else {
                oracle_target_probs(row, V, (double)tau, p);
                double pt = p[x[i]];
                double qt = (double)qrows[(size_t)i * V + x[i]];
                accept = ((double)u[i] * qt < pt);
                if (qt > 0.0) {
                    ratio = pt / qt < 1.0 ? pt / qt : 1.0;
                    m = fabs((double)u[i] - pt / qt);
                } else {
                    ratio = 1.0;
                }
            }
            if (accept_ratio)
                accept_ratio[(size_t)b * k + i] = ratio;
            if (j == k) {
                if (mg)
                    mg[i] = m;
                if (!accept)
                    j = i;
            }
        }

        /* The token at position j: corrected (j < k) or bonus (j == k). */
        int final_token;
        const float *row_j = rows + (size_t)j * V;
        if (greedy) {
            final_token = oracle_argmax(row_j, V);
        } else {
            oracle_target_probs(row_j, V, (double)tau, p);
            double mass = 0.0;
            if (j < k) {
                const float *qj = qrows + (size_t)j * V;
                for (int y = 0; y < V; ++y) {
                    double diff = p[y] - (double)qj[y];
                    r[y] = diff > 0.0 ? diff : 0.0;
                    mass += r[y];
                }
            }
            if (j == k || !(mass > 0.0)) {
                mass = 0.0;
                for (int y = 0; y < V; ++y) {
                    r[y] = p[y];
                    mass += r[y];
                }
            }
            const double target = (double)u[k] * mass;
            double cdf = 0.0;
            double nearest = INFINITY;
            final_token = -1;
            int last_positive = -1;
            for (int y = 0; y < V; ++y) {
                cdf += r[y];
                if (r[y] > 0.0)
                    last_positive = y;
                double dist = fabs((double)u[k] - cdf / mass);
                if (dist < nearest)
                    nearest = dist;
                if (final_token < 0 && target < cdf)
                    final_token = y;
            }
            if (final_token < 0)
                final_token = last_positive;
            if (mg)
                mg[k] = nearest;
        }

        num_accepted[b] = j;
        int32_t *ob = out_tokens + (size_t)b * (k + 1);
        for (int i = 0; i <= k; ++i)
            ob[i] = -1;
        for (int i = 0; i < j; ++i)
            ob[i] = x[i];
        ob[j] = final_token;
    }
    free(p);
    free(r);
    return ORACLE_OK;
}

/*
 * 4. KV commit after acceptance (Sec. 3.1: the accepted candidates join the
 *    context and generation continues from the first rejected position;
 *    Sec. 3.3: the next draft block starts from the emitted token).
 *
 *    Reading adopted (the paper gives no cache mechanics): the n_q rows
 *    verified for sequence b sit at cache positions L_b .. L_b + n_q - 1,
 *    L_b = seq_lens[b] - n_q, and row i belongs to the i-th token of the
 *    verified block, whose first token is the previously emitted one.  With
 *    a = num_accepted[b] drafts accepted, the first keep = min(a + 1, n_q)
 *    rows stay valid and the rest are dropped: the cached length becomes
 *    L'_b = L_b + keep.  The next verification of n_q_next rows writes them
 *    at L'_b .., so seq_lens[b] becomes L'_b + n_q_next, and the block table
 *    must map exactly need_b = ceil(seq_lens[b] / page_size) logical pages
 *    (it mapped ceil(old seq_lens[b] / page_size) before).
 *
 *    Page bookkeeping through a stack of free physical pages
 *    free_pages[0 .. *free_count):
 *      1. for b = 0 .. B-1, for each logical page lp = need_b .. had_b - 1
 *         (ascending): push block_table[b][lp] and set the entry to -1;
 *      2. then for b = 0 .. B-1, for each logical page lp = had_b ..
 *         need_b - 1 (ascending): take the stack entry at index
 *         (top after step 1) - (total pages taken) + (count taken so far),
 *         i.e. the taken pages are the topmost entries, assigned bottom-up;
 *      3. the stack keeps its entries below that point.
 *    All or nothing: if any sequence is invalid (seq_lens[b] < n_q,
 *    num_accepted[b] < 0, need_b > max_pages) the result is
 *    ORACLE_ERR_ARG, and if the stack would overflow `capacity` or run out
 *    of pages it is ORACLE_ERR_PAGES; in both cases nothing is modified.
 */
#define ORACLE_ERR_PAGES 5

/* Cached length for the next step and logical pages before / after. */
static void commit_plan(int T, int a, int n_q, int n_q_next, int page_size, long long *next_len,
                        long long *had, long long *need)
{
    const int keep = a + 1 < n_q ? a + 1 : n_q;
    *next_len = (long long)(T - n_q) + keep + n_q_next;
    *had = ((long long)T + page_size - 1) / page_size;
    *need = (*next_len + page_size - 1) / page_size;
}

int oracle_kv_commit(int32_t *seq_lens, int32_t *block_table, int32_t *free_pages,
                     int32_t *free_count, const int32_t *num_accepted, int B, int n_q,
                     int n_q_next, int max_pages, int page_size, int capacity)
{
    if (B < 1 || n_q < 1 || n_q_next < 1 || max_pages < 1 || page_size < 1 || capacity < 0 ||
        *free_count < 0 || *free_count > capacity)
        return ORACLE_ERR_ARG;
    long long pushed = 0, taken = 0, next_len, had, need;
    for (int b = 0; b < B; ++b) {
        if (seq_lens[b] < n_q || num_accepted[b] < 0)
            return ORACLE_ERR_ARG;
        commit_plan(seq_lens[b], num_accepted[b], n_q, n_q_next, page_size, &next_len, &had,
                    &need);
        if (need > max_pages || had > max_pages)
            return ORACLE_ERR_ARG;
        if (need < had)
            pushed += had - need;
        else
            taken += need - had;
    }
    const long long top = (long long)*free_count + pushed;
    if (top > capacity || taken > top)
        return ORACLE_ERR_PAGES;

    /* step 1: surplus pages onto the stack, in sequence order */
    long long sp = *free_count;
    for (int b = 0; b < B; ++b) {
        commit_plan(seq_lens[b], num_accepted[b], n_q, n_q_next, page_size, &next_len, &had,
                    &need);
        int32_t *row = block_table + (size_t)b * max_pages;
        for (long long lp = need; lp < had; ++lp) {
            free_pages[sp++] = row[lp];
            row[lp] = -1;
        }
    }
    /* step 2: missing pages from the top `taken` stack entries, bottom-up */
    long long take = top - taken;
    for (int b = 0; b < B; ++b) {
        commit_plan(seq_lens[b], num_accepted[b], n_q, n_q_next, page_size, &next_len, &had,
                    &need);
        int32_t *row = block_table + (size_t)b * max_pages;
        for (long long lp = had; lp < need; ++lp)
            row[lp] = free_pages[take++];
        seq_lens[b] = (int32_t)next_len;
    }
    *free_count = (int32_t)(top - taken);
    return ORACLE_OK;
}

/*
 * 5. Draft tail sampling (Algorithm 1, last two steps: the LM head turns the
 *    semi-autoregressive head's K hidden states into distributions
 *    P'_1..P'_K, and T'_i ~ Categorical(P'_i); Sec. 3.3).  Given the fp32
 *    logits of R rows: P' = softmax(logits / tau) (tau = the row's draft
 *    temperature), and the token is drawn by inverse CDF with the row's
 *    uniform u: the smallest x (ascending token id) with u * S < C(x),
 *    C(x) = sum_{y <= x} exp((l_y - m) / tau), S = C(V - 1) (the same
 *    convention as the residual draw of the acceptance); if rounding leaves
 *    none, the last x with non-zero weight.  tau <= 0 is greedy drafting:
 *    the token is the first argmax of the raw logits and P' is one-hot on it
 *    (the limit of the softmax as tau -> 0 for a unique maximum).
 *    margin[r] = min_x |u - C(x) / S| (0 for greedy rows): the distance of
 *    the draw to the nearest CDF boundary.
 */
int oracle_sample(const float *logits, const float *uniforms, const float *temperature, int R,
                  int V, double *probs, int32_t *tokens, double *margin)
{
    if (R < 1 || V < 1)
        return ORACLE_ERR_ARG;
    for (int r = 0; r < R; ++r) {
        const float *row = logits + (size_t)r * V;
        double *pr = probs + (size_t)r * V;
        const double tau = temperature[r];
        int best = 0;
        for (int x = 1; x < V; ++x)
            if (row[x] > row[best])
                best = x;
        if (!(tau > 0.0)) {
            for (int x = 0; x < V; ++x)
                pr[x] = 0.0;
            pr[best] = 1.0;
            tokens[r] = best;
            if (margin)
                margin[r] = 0.0;
            continue;
        }
        const double m = (double)row[best] / tau;
        double S = 0.0;
        for (int x = 0; x < V; ++x) {
            pr[x] = exp((double)row[x] / tau - m);
            S += pr[x];
        }
        const double u = uniforms[r];
        const double target = u * S;
        double cdf = 0.0, nearest = INFINITY;
        int tok = -1, last_positive = -1;
        for (int x = 0; x < V; ++x) {
            cdf += pr[x];
            if (pr[x] > 0.0)
                last_positive = x;
            const double dist = fabs(u - cdf / S);
            if (dist < nearest)
                nearest = dist;
            if (tok < 0 && target < cdf)
                tok = x;
        }
        if (tok < 0)
            tok = last_positive;
        for (int x = 0; x < V; ++x)
            pr[x] /= S;
        tokens[r] = tok;
        if (margin)
            margin[r] = nearest;
    }
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------ */
/* Visual token compression (Sec. 3.2, Eq. 3; Algorithm 1): the draft model */
/* compresses the N visual features F_V of an image or frame into C          */
/* features with a learnable query set Q (C x d):                             */
/*     F^_V = softmax(Q F_V^T) F_V,                                           */
/* F_V serving as both keys and values.  Readings: the softmax runs over the */
/* N visual tokens of one query (its weights sum to 1), the scores are not   */
/* scaled (Eq. 3 writes none), and a clip of F frames is F independent        */
/* images of N tokens each sharing the same queries.                          */
/*                                                                            */
/* queries   bf16 bits [C][d]                                                 */
/* features  bf16 bits [F][N][d]                                              */
/* out       [F][C][d] doubles                                                */
/* ------------------------------------------------------------------------ */
int oracle_visual_compress(const uint16_t *queries, const uint16_t *features, int F, int N, int C,
                           int d, double *out)
{
    if (F < 1 || N < 1 || C < 1 || d < 1)
        return ORACLE_ERR_ARG;
    double *s = (double *)malloc(sizeof(double) * (size_t)N);
    if (!s)
        return ORACLE_ERR_NOMEM;
    for (int f = 0; f < F; ++f) {
        const uint16_t *fv = features + (size_t)f * N * d;
        for (int c = 0; c < C; ++c) {
            const uint16_t *qc = queries + (size_t)c * d;
            /* scores of query c against every token of the frame */
            double smax = -INFINITY;
            for (int n = 0; n < N; ++n) {
                double acc = 0.0;
                for (int j = 0; j < d; ++j)
                    acc += oracle_bf16_value(qc[j]) * oracle_bf16_value(fv[(size_t)n * d + j]);
                s[n] = acc;
                if (acc > smax)
                    smax = acc;
            }
            /* softmax over the tokens */
            double z = 0.0;
            for (int n = 0; n < N; ++n) {
                s[n] = exp(s[n] - smax);
                z += s[n];
            }
            /* weighted sum of the token features */
            double *o = out + ((size_t)f * C + c) * d;
            for (int j = 0; j < d; ++j)
                o[j] = 0.0;
            for (int n = 0; n < N; ++n) {
                const double w = s[n] / z;
                for (int j = 0; j < d; ++j)
                    o[j] += w * oracle_bf16_value(fv[(size_t)n * d + j]);
            }
        }
    }
    free(s);
    return ORACLE_OK;
}

/* Threads of the OpenMP loops (the per-row attention loop): n >= 1 sets the
 * count, n <= 0 restores the default.  Every result is independent of it
 * (each row is computed by one thread in a fixed order); bench.py times the
 * oracle on one thread and on all host cores. */
void oracle_set_threads(int n)
{
    omp_set_num_threads(n >= 1 ? n : omp_get_num_procs());
}
