/*
 * hsa_oracle.c -- plain, slow CPU oracle of the Heterogeneous Step Allocation
 * (HSA) hot path.
 *
 * TEST INFRASTRUCTURE.  Only the test-suite, the package smoke check and the
 * benchmark's CPU-baseline leg load this file.  The CUDA library never calls
 * it, includes nothing from it, and it includes nothing from the library: the
 * two sides share no header, helper, table or constant.
 *
 * Every routine is the paper's definition written out directly, in fp64
 * unless stated otherwise, with no blocking, fusion or reordering:
 *
 *   orc_partition        Sec. 2.2 Eq. 3 and the divisor constraint (Eq. 5),
 *                        ranked as App. B "dynamic token selection" (Eq. 7):
 *                        a smaller statistic goes to a lower-budget group.
 *   orc_margin/is_active Sec. 2.2 modular activity rule (after Eq. 5) and Sec. 2.5
 *                        "phase-aware caching window".
 *   orc_active_set       Sec. 2.3 active set A_i (ascending token order).
 *   orc_gather           Sec. 2.3 step 1, the rows x[A_i] entering the block.
 *   orc_kv_scatter       Sec. 2.3 step 2, cache update K^[A_i] <- K[A_i].
 *   orc_attention        Sec. 2.3 step 3, active queries against the full cache.
 *   orc_cached_euler_*   Sec. 2.4 Eq. 6 (cached Euler update), with the
 *                        velocity cache refreshed for active tokens.
 *   orc_sigmas           Sec. 2.1 noise schedule of the Euler solver (Eq. 2).
 *   orc_l1rel_accumulate App. B Eq. 7, the per-token L1 relative change of the
 *                        velocity, accumulated (weighted) into a running mean.
 *   orc_uniform_stat     App. B "uniform allocation (U)": a statistic whose
 *                        ranking gives every group evenly spread positions.
 *   orc_reserve_frame    App. B "first-frame reservation (F)".
 *   orc_reorder          Sec. 2.5 "token reordering": non-baseline tokens
 *                        first, then the baseline group, each in token order.
 *   orc_rope_table,      Sec. 2.3: rotary position embedding of the active
 *   orc_rope_rows        rows, their frequencies subsampled (gathered) to A_i.
 *
 * Readings where the paper is silent (each is listed with its reason in the
 * design notes): ties in the ranking go to the lower token index first and
 * -0 equals +0; a non-finite statistic is an error; the window margin is the
 * integer floor((100-k)*T/200) with k in percent; the softmax scale defaults
 * to 1/sqrt(D) with no mask; group ids are 0-based, group 0 the baseline; an
 * L1 relative change with a zero denominator is 0 when the numerator is 0 and
 * the largest finite fp32 value otherwise.
 *
 * Status codes (plain ints): 0 ok, -1 invalid argument, -2 a budget does not
 * divide T, -3 counts do not sum to N, -5 non-finite statistic, -6 index
 * out of range or duplicated.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_EINVAL (-1)
#define ORC_ENOTDIV (-2)
#define ORC_ECOUNTS (-3)
#define ORC_ENONFINITE (-5)
#define ORC_EINDEX (-6)

/* ---------------------------------------------------------------- budgets */

/* Budgets must satisfy Sec. 2.2: s_1 = T (baseline), s_1 >= s_2 >= ... >= s_K,
 * every s_k a positive divisor of T; counts |G_k| >= 0 with sum N. */
int orc_check_budgets(int T, const int *budgets, const int *counts, int K, int N)
{
    if (T < 1 || K < 1 || N < 0 || !budgets)
        return ORC_EINVAL;
    for (int k = 0; k < K; ++k) {
        if (budgets[k] < 1 || budgets[k] > T)
            return ORC_EINVAL;
        if (T % budgets[k] != 0)
            return ORC_ENOTDIV;
        if (k > 0 && budgets[k] > budgets[k - 1])
            return ORC_EINVAL;
    }
    if (budgets[0] != T)
        return ORC_EINVAL;
    if (counts) {
        long long sum = 0;
        for (int k = 0; k < K; ++k) {
            if (counts[k] < 0)
                return ORC_ECOUNTS;
            sum += counts[k];
        }
        if (sum != N)
            return ORC_ECOUNTS;
    }
    return ORC_OK;
}

/* -------------------------------------------------------------- partition */

static const float *g_sort_stat; /* qsort has no context argument */

/* Order of tokens by (statistic ascending, index ascending).  Comparing the
 * floats with < makes -0 and +0 equal, so such ties fall to the index. */
static int cmp_token(const void *pa, const void *pb)
{
    int a = *(const int *)pa, b = *(const int *)pb;
    float va = g_sort_stat[a], vb = g_sort_stat[b];
    if (va < vb) return -1;
    if (vb < va) return 1;
    return (a > b) - (a < b);
}

/* Token partition (Sec. 2.2 Eq. 3) by ranking the per-token statistic
 * (App. B, Eq. 7): the |G_K| tokens with the smallest statistic go to the
 * smallest budget s_K, the next |G_{K-1}| to s_{K-1}, ..., the |G_1| largest
 * to the baseline group.  Writes group_of[n] in [0, K), group 0 = baseline. */
int orc_partition(const float *stat, int N, int T, const int *budgets,
                  const int *counts, int K, int32_t *group_of)
{
    int st = orc_check_budgets(T, budgets, counts, K, N);
    if (st != ORC_OK)
        return st;
    if (!counts || (N > 0 && (!stat || !group_of)))
        return ORC_EINVAL;
    for (int n = 0; n < N; ++n)
        if (!isfinite(stat[n]))
            return ORC_ENONFINITE;
    int *order = (int *)malloc(sizeof(int) * (size_t)(N > 0 ? N : 1));
    if (!order)
        return ORC_EINVAL;
    for (int n = 0; n < N; ++n)
        order[n] = n;
    g_sort_stat = stat;
    qsort(order, (size_t)N, sizeof(int), cmp_token);
    int r = 0;
    for (int k = K - 1; k >= 0; --k)
        for (int c = 0; c < counts[k]; ++c, ++r)
            group_of[order[r]] = k;
    free(order);
    return ORC_OK;
}

/* ----------------------------------------------------------- active sets */

/* Caching-window margin m = floor((1-k) T / 2) of Sec. 2.5, k = window_pct/100,
 * computed in integers so that e.g. k = 80%, T = 40 gives exactly 4. */
int orc_margin(int T, int window_pct)
{
    if (T < 1 || window_pct < 0 || window_pct > 100)
        return ORC_EINVAL;
    return ((100 - window_pct) * T) / 200;
}

/* Group with budget s is active at global iteration i iff i mod (T/s) == 0
 * (Sec. 2.2), or i lies outside the caching window [m, T-m-1] (Sec. 2.5). */
int orc_is_active(int i, int T, int s, int m)
{
    if (i < m || i > T - m - 1)
        return 1;
    return (i % (T / s)) == 0;
}

/* Active set A_i (Sec. 2.3): every token whose group is active at iteration
 * iter, in ascending token order; pos[n] = rank of n in A_i, or -1 when n is
 * skipped (pos may be NULL).  Returns |A_i| or a negative status. */
int orc_active_set(const int32_t *group_of, int N, int T, const int *budgets,
                   int K, int iter, int window_pct, int32_t *idx, int32_t *pos)
{
    int st = orc_check_budgets(T, budgets, NULL, K, N);
    if (st != ORC_OK)
        return st;
    int m = orc_margin(T, window_pct);
    if (m < 0 || iter < 0 || iter >= T)
        return ORC_EINVAL;
    int cnt = 0;
    for (int n = 0; n < N; ++n) {
        int g = group_of[n];
        if (g < 0 || g >= K)
            return ORC_EINDEX;
        if (orc_is_active(iter, T, budgets[g], m)) {
            if (idx)
                idx[cnt] = n;
            if (pos)
                pos[n] = cnt;
            ++cnt;
        } else if (pos) {
            pos[n] = -1;
        }
    }
    return cnt;
}

/* |A_i| from the group sizes alone. */
int orc_active_count(const int *budgets, const int *counts, int K, int T,
                     int iter, int window_pct)
{
    int m = orc_margin(T, window_pct);
    if (m < 0)
        return m;
    long long cnt = 0;
    for (int k = 0; k < K; ++k)
        if (orc_is_active(iter, T, budgets[k], m))
            cnt += counts[k];
    return (int)cnt;
}

/* ------------------------------------------------------ gather / scatter */

static int check_idx(const int32_t *idx, int n_active, int N)
{
    for (int j = 0; j < n_active; ++j)
        if (idx[j] < 0 || idx[j] >= N)
            return ORC_EINDEX;
    return ORC_OK;
}

/* dst[j, :] = src[idx[j], :] (Sec. 2.3 step 1: only x[A_i] enters the block). */
int orc_gather(const void *src, size_t row_bytes, int N, const int32_t *idx,
               int n_active, void *dst)
{
    if (check_idx(idx, n_active, N))
        return ORC_EINDEX;
    for (int j = 0; j < n_active; ++j)
        memcpy((char *)dst + (size_t)j * row_bytes,
               (const char *)src + (size_t)idx[j] * row_bytes, row_bytes);
    return ORC_OK;
}

/* K^[idx[j]] = K[j], V^[idx[j]] = V[j] (Sec. 2.3 step 2); rows of skipped
 * tokens are left as they are.  Duplicate indices are rejected because the
 * groups are disjoint (Sec. 2.2), so A_i never repeats a token. */
int orc_kv_scatter(void *k_cache, void *v_cache, const void *k_fresh,
                   const void *v_fresh, const int32_t *idx, int n_active,
                   int N, size_t row_bytes)
{
    if (check_idx(idx, n_active, N))
        return ORC_EINDEX;
    char *seen = (char *)calloc((size_t)(N > 0 ? N : 1), 1);
    if (!seen)
        return ORC_EINVAL;
    for (int j = 0; j < n_active; ++j) {
        if (seen[idx[j]]) {
            free(seen);
            return ORC_EINDEX;
        }
        seen[idx[j]] = 1;
    }
    free(seen);
    for (int j = 0; j < n_active; ++j) {
        memcpy((char *)k_cache + (size_t)idx[j] * row_bytes,
               (const char *)k_fresh + (size_t)j * row_bytes, row_bytes);
        memcpy((char *)v_cache + (size_t)idx[j] * row_bytes,
               (const char *)v_fresh + (size_t)j * row_bytes, row_bytes);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------- attention */

/* Element of a tensor stored as bf16 (dtype 0), fp32 (1) or fp64 (2),
 * widened exactly to fp64. */
static double elem(const void *p, int dtype, size_t i)
{
    if (dtype == 0) {
        uint32_t u = (uint32_t)((const uint16_t *)p)[i] << 16;
        float f;
        memcpy(&f, &u, sizeof f);
        return (double)f;
    }
    if (dtype == 1)
        return (double)((const float *)p)[i];
    return ((const double *)p)[i];
}

/* Full-context attention of the active queries (Sec. 2.3 step 3):
 *   out[j,h,:] = sum_n softmax_n(scale * <q_{r,h}, k^_{n,h}>) v^_{n,h}
 * over all N cached keys, r = q_idx[j] (q is [rows, H, D]) or r = j when
 * q_idx is NULL (q is compact [n_q, H, D]).  K^, V^ are [N, H, D].  The
 * softmax subtracts the row maximum before exp, which leaves it unchanged.
 * scale <= 0 selects 1/sqrt(D).  out is fp64 [n_q, H, D]. */
int orc_attention(const void *q, int q_dtype, const int32_t *q_idx, int n_q,
                  const void *k, const void *v, int kv_dtype, int N, int H,
                  int D, double scale, double *out)
{
    if (N < 1 || H < 1 || D < 1 || n_q < 0)
        return ORC_EINVAL;
    if (scale <= 0.0)
        scale = 1.0 / sqrt((double)D);
    double *s = (double *)malloc(sizeof(double) * (size_t)N);
    if (!s)
        return ORC_EINVAL;
    for (int j = 0; j < n_q; ++j) {
        size_t r = q_idx ? (size_t)q_idx[j] : (size_t)j;
        for (int h = 0; h < H; ++h) {
            size_t qo = (r * (size_t)H + (size_t)h) * (size_t)D;
            double mx = -INFINITY;
            for (int n = 0; n < N; ++n) {
                size_t ko = ((size_t)n * (size_t)H + (size_t)h) * (size_t)D;
                double dot = 0.0;
                for (int d = 0; d < D; ++d)
                    dot += elem(q, q_dtype, qo + (size_t)d) * elem(k, kv_dtype, ko + (size_t)d);
                s[n] = scale * dot;
                if (s[n] > mx)
                    mx = s[n];
            }
            double l = 0.0;
            for (int n = 0; n < N; ++n) {
                s[n] = exp(s[n] - mx);
                l += s[n];
            }
            double *o = out + ((size_t)j * (size_t)H + (size_t)h) * (size_t)D;
            for (int d = 0; d < D; ++d)
                o[d] = 0.0;
            for (int n = 0; n < N; ++n) {
                size_t vo = ((size_t)n * (size_t)H + (size_t)h) * (size_t)D;
                for (int d = 0; d < D; ++d)
                    o[d] += s[n] * elem(v, kv_dtype, vo + (size_t)d);
            }
            for (int d = 0; d < D; ++d)
                o[d] /= l;
        }
    }
    free(s);
    return ORC_OK;
}

/* ----------------------------------------------------------- cached Euler */

/* Cached Euler update (Sec. 2.4 Eq. 6) over all N tokens, fp64:
 * for an active token (pos[n] >= 0) the velocity cache first takes the fresh
 * velocity, v^[n] <- v_fresh[pos[n]]; then every token advances
 * x[n] <- x[n] + v^[n] * dsigma, dsigma = sigma_{i+1} - sigma_i.
 * v_fresh and pos may both be NULL (no token refreshed). */
int orc_cached_euler_f64(double *x, double *vhat, const double *v_fresh,
                         const int32_t *pos, int N, int C, double dsigma)
{
    for (int n = 0; n < N; ++n) {
        if (pos && pos[n] >= 0) {
            if (!v_fresh)
                return ORC_EINVAL;
            for (int c = 0; c < C; ++c)
                vhat[(size_t)n * C + c] = v_fresh[(size_t)pos[n] * C + c];
        }
        for (int c = 0; c < C; ++c)
            x[(size_t)n * C + c] = x[(size_t)n * C + c] + vhat[(size_t)n * C + c] * dsigma;
    }
    return ORC_OK;
}

/* The same update in fp32: dsigma is the fp64 difference rounded once to
 * fp32, and each element takes one fused multiply-add (a single rounding). */
int orc_cached_euler_f32(float *x, float *vhat, const float *v_fresh,
                         const int32_t *pos, int N, int C, float dsigma)
{
    for (int n = 0; n < N; ++n) {
        if (pos && pos[n] >= 0) {
            if (!v_fresh)
                return ORC_EINVAL;
            for (int c = 0; c < C; ++c)
                vhat[(size_t)n * C + c] = v_fresh[(size_t)pos[n] * C + c];
        }
        for (int c = 0; c < C; ++c)
            x[(size_t)n * C + c] = fmaf(vhat[(size_t)n * C + c], dsigma, x[(size_t)n * C + c]);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------- schedules */

/* sigma_i, i = 0..T, decreasing from 1 to sigma_T = 0 (Sec. 2.1).  shift = 1
 * is the linear schedule sigma_i = 1 - i/T; shift s != 1 applies the
 * flow-matching time shift sigma = s t / (1 + (s-1) t) to t_i = 1 - i/T. */
int orc_sigmas(int T, double shift, double *sigma)
{
    if (T < 1 || !(shift > 0.0))
        return ORC_EINVAL;
    for (int i = 0; i <= T; ++i) {
        double t = 1.0 - (double)i / (double)T;
        sigma[i] = shift * t / (1.0 + (shift - 1.0) * t);
    }
    return ORC_OK;
}

/* ------------------------------------------------- velocity statistic (D) */

/* App. B Eq. 7: for every token refreshed at this step (pos[n] >= 0),
 *   L1rel(n, i) = ||v_i[n] - v_{i-1}[n]||_1 / ||v_i[n]||_1
 * with v_i[n] = v_fresh[pos[n]] and v_{i-1}[n] = vhat_old[n] (the velocity
 * cache before this step's refresh), and stat[n] += weight * L1rel(n, i).
 * With weight = 1/(number of averaged steps) stat ends as the mean over the
 * initial full-budget steps, the statistic the dynamic selection ranks. */
int orc_l1rel_accumulate(const double *vhat_old, const double *v_fresh, const int32_t *pos,
                         int N, int C, double weight, double *stat)
{
    for (int n = 0; n < N; ++n) {
        if (!pos || pos[n] < 0)
            continue;
        const double *vn = v_fresh + (size_t)pos[n] * C;
        const double *vo = vhat_old + (size_t)n * C;
        double num = 0.0, den = 0.0;
        for (int c = 0; c < C; ++c) {
            num += fabs(vn[c] - vo[c]);
            den += fabs(vn[c]);
        }
        double r;
        if (den == 0.0)
            r = (num == 0.0) ? 0.0 : 3.4028234663852886e38;
        else
            r = num / den;
        stat[n] += weight * r;
    }
    return ORC_OK;
}

/* -------------------------------------------------- allocation strategies */

/* Uniform allocation (App. B, U).  Reading: token n gets the statistic
 * floor(frac((n+1) * phi) * 2^24) with phi = (sqrt(5)-1)/2, taken as the top
 * 24 bits of the 32-bit product (n+1) * 2654435769 (= round(phi * 2^32)).
 * Ranking it (orc_partition) gives each group the tokens whose value lies in
 * one interval of the circle, which by the three-distance theorem are spaced
 * by at most three distinct gaps: maximally spread over the sequence. */
int orc_uniform_stat(int N, float *stat)
{
    for (int n = 0; n < N; ++n) {
        uint32_t h = (uint32_t)(n + 1) * 2654435769u;
        stat[n] = (float)(h >> 8);
    }
    return ORC_OK;
}

/* First-frame reservation (App. B, F): the first frame_tokens tokens (frame 0
 * in row-major token order) get the largest finite fp32 statistic, so a
 * ranking places them in the baseline group when |G_1| >= frame_tokens. */
int orc_reserve_frame(float *stat, int N, int frame_tokens)
{
    if (frame_tokens < 0 || frame_tokens > N)
        return ORC_EINVAL;
    for (int n = 0; n < frame_tokens; ++n)
        stat[n] = 3.40282347e38f;
    return ORC_OK;
}

/* ------------------------------------------------------- token reordering */

/* Token reordering (Sec. 2.5): new position r holds old token order[r]; the
 * tokens of groups 1..K-1 come first in their original order, then the
 * baseline group 0 in its original order.  where[n] is the new position of
 * old token n (the inverse permutation, used to undo the reordering), and
 * group_new[r] = group_of[order[r]].  Returns the number of non-baseline
 * tokens M (the length of the cached prefix). */
int orc_reorder(const int32_t *group_of, int N, int32_t *order, int32_t *where,
                int32_t *group_new)
{
    int r = 0;
    for (int n = 0; n < N; ++n)
        if (group_of[n] != 0) {
            order[r] = n;
            where[n] = r;
            group_new[r] = group_of[n];
            ++r;
        }
    const int M = r;
    for (int n = 0; n < N; ++n)
        if (group_of[n] == 0) {
            order[r] = n;
            where[n] = r;
            group_new[r] = 0;
            ++r;
        }
    return M;
}

/* ------------------------------------------------------------- rotary (RoPE) */

/* Rotary embedding table of a (F, Hh, Ww) token grid, tokens row-major over
 * (f, h, w).  Reading (the paper names RoPE but not its layout): the D/2
 * rotation pairs are split into three bands, p_h = p_w = floor(D/6) pairs for
 * the row and column axes and p_t = D/2 - 2*p_h for the frame axis, in that
 * order (t, h, w); pair i of a band with p pairs turns by
 * pos * theta^(-i/p).  table[n][i] = (cos, sin) of token n's angle for pair
 * i, computed in fp64 and rounded to fp32 (the table's storage type). */
int orc_rope_table(int F, int Hh, int Ww, int D, double theta, float *table)
{
    if (F < 1 || Hh < 1 || Ww < 1 || D < 2 || (D & 1) || !(theta > 1.0))
        return ORC_EINVAL;
    const int P = D / 2, ph = D / 6, pt = P - 2 * (D / 6);
    for (int f = 0; f < F; ++f)
        for (int h = 0; h < Hh; ++h)
            for (int w = 0; w < Ww; ++w) {
                const size_t n = ((size_t)f * Hh + h) * Ww + w;
                for (int i = 0; i < P; ++i) {
                    int band_i, band_p, pos;
                    if (i < pt) {
                        band_i = i; band_p = pt; pos = f;
                    } else if (i < pt + ph) {
                        band_i = i - pt; band_p = ph; pos = h;
                    } else {
                        band_i = i - pt - ph; band_p = ph; pos = w;
                    }
                    const double ang = pos * pow(theta, -(double)band_i / band_p);
                    table[(n * P + i) * 2] = (float)cos(ang);
                    table[(n * P + i) * 2 + 1] = (float)sin(ang);
                }
            }
    return ORC_OK;
}

static uint16_t to_bf16(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7fffffffu) > 0x7f800000u)
        return (uint16_t)((u >> 16) | 0x40u);          /* NaN stays NaN */
    u += 0x7fffu + ((u >> 16) & 1u);                    /* round to nearest even */
    return (uint16_t)(u >> 16);
}

/* Rotate rows j < n of a bf16 tensor x[n][H][D] in place by the table row of
 * their token idx[j] (the frequencies subsampled to the active set):
 * (x0, x1) -> (x0 c - x1 s, x0 s + x1 c) per pair, as
 * y0 = fma(x0, c, -(x1 s)), y1 = fma(x0, s, x1 c) in fp32, rounded to bf16. */
int orc_rope_rows(uint16_t *x, const int32_t *idx, int n, int H, int D, const float *table,
                  int N)
{
    const int P = D / 2;
    for (int j = 0; j < n; ++j) {
        if (idx[j] < 0 || idx[j] >= N)
            return ORC_EINDEX;
        const float *t = table + (size_t)idx[j] * P * 2;
        for (int h = 0; h < H; ++h) {
            uint16_t *row = x + ((size_t)j * H + h) * D;
            for (int i = 0; i < P; ++i) {
                uint32_t a = (uint32_t)row[2 * i] << 16, b = (uint32_t)row[2 * i + 1] << 16;
                float x0, x1;
                memcpy(&x0, &a, 4);
                memcpy(&x1, &b, 4);
                const float c = t[2 * i], s = t[2 * i + 1];
                const float y0 = fmaf(x0, c, -(x1 * s));
                const float y1 = fmaf(x0, s, x1 * c);
                row[2 * i] = to_bf16(y0);
                row[2 * i + 1] = to_bf16(y1);
            }
        }
    }
    return ORC_OK;
}
