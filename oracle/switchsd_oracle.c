/*
 * switchsd_oracle.c -- plain, slow CPU oracle of the SwitchSD per-step controller.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the reference the CUDA path is checked against.  Only the
 * test suite, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load it.  It shares no code,
 * header, table or constant with the CUDA library (paper_2609_20186_gb300/csrc), and it includes
 * nothing from there.  Every function follows one passage of the paper ("To Copy or Not to Copy:
 * Controlling Speculative Decoding via Intrinsic Model Signals"), cited beside it, and is written as the
 * plain definition: no blocking, no early reordering, floating point in double.
 *
 * Conventions (shared with the CUDA path only through the documented C ABI, not through code):
 *   - a context row is int32 tokens x[0..L-1]; the current token is x[L-1];
 *   - bf16 values arrive as their 16-bit patterns (uint16_t);
 *   - modes: 0 = no repetition, 1 = copy draft, 2 = repetition without copy intent (Fig. 1 cases i-iii).
 *
 * Parity status: every function below is pinned by tests that do not re-run its own formula
 * (brute-force enumeration, hand-built cases, library routines, closed forms); see tests/test_oracle_*.py.
 */
#include <stdint.h>
#include <string.h>

#define ORACLE_MODE_NO_REP 0
#define ORACLE_MODE_COPY 1
#define ORACLE_MODE_REP_NO_COPY 2

#define ORACLE_ROW_OK 0
#define ORACLE_ROW_CAPACITY 1

/*
 * Longest-suffix n-gram search.  §3.3 "Copy-Intent Decision Rule": the n-gram ending at the current
 * token x_i must match a prior occurrence in the context; §3.3 "Copy-Based Speculative Generation":
 * candidates are ranked by recency.  Reading of the open points: n is tried from n_max down to n_min
 * and the first n with an occurrence wins; for that n the most recent occurrence (largest end e) wins;
 * a prior occurrence ends at e <= L-2 so that at least one continuation token exists; occurrences may
 * overlap the suffix itself.
 * Returns 1 with (*n_out, *e_out) on a hit, else 0 with (0, -1).
 */
int oracle_longest_suffix_match(const int32_t *x, int32_t L, int32_t n_min, int32_t n_max,
                                int32_t *n_out, int32_t *e_out)
{
    for (int32_t n = n_max; n >= n_min; --n) {
        if (L < n + 1) continue;               /* the suffix and one earlier end must both fit */
        for (int32_t e = L - 2; e >= n - 1; --e) {
            int32_t i = 0;
            while (i < n && x[e - i] == x[L - 1 - i]) ++i;
            if (i == n) {
                *n_out = n;
                *e_out = e;
                return 1;
            }
        }
    }
    *n_out = 0;
    *e_out = -1;
    return 0;
}

/* bf16 bit pattern -> double: a bf16 is the upper half of an IEEE binary32. */
double oracle_bf16_to_double(uint16_t v)
{
    uint32_t bits = ((uint32_t)v) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/*
 * Linear copy-intent probe, Eq. 3: p = sigma(w^T H), no bias.  The oracle returns the logit
 * z = w^T H, summed in double in index order.
 */
double oracle_probe_linear(const uint16_t *h, const uint16_t *w, int32_t d)
{
    double z = 0.0;
    for (int32_t j = 0; j < d; ++j)
        z += oracle_bf16_to_double(w[j]) * oracle_bf16_to_double(h[j]);
    return z;
}

/*
 * Two-layer probe z = w2 . ReLU(W1 h + b1) + b2 (an extension beyond Eq. 3's linear probe, used by
 * the 256-row / 5120-wide workload).  W1 is [H1, d] row-major bf16, w2 is [H1] bf16, b1 is [H1] float
 * or NULL, b2 a float.  All arithmetic in double; the hidden layer is never rounded.
 */
double oracle_probe_mlp(const uint16_t *h, const uint16_t *W1, const float *b1, const uint16_t *w2,
                        float b2, int32_t d, int32_t H1)
{
    double z = (double)b2;
    for (int32_t u = 0; u < H1; ++u) {
        double a = (b1 != NULL) ? (double)b1[u] : 0.0;
        for (int32_t j = 0; j < d; ++j)
            a += oracle_bf16_to_double(W1[(int64_t)u * d + j]) * oracle_bf16_to_double(h[j]);
        if (a < 0.0) a = 0.0;
        z += oracle_bf16_to_double(w2[u]) * a;
    }
    return z;
}

/*
 * Three-way switch and copy draft.  Fig. 1: (i) no repetition -> neural draft; (ii) repetition with
 * copy intent -> copy draft; (iii) repetition without copy intent -> neural draft.  Eq. 4 and the
 * kappa-gram condition of §3.3: copy iff sigma(z) >= tau and the kappa-gram ending at x_{L-1} occurs
 * earlier.  Since sigma is monotone, sigma(z) >= tau is decided as z >= logit(tau); the comparison is
 * taken in binary32, the precision the device path decides in.  A match shorter than kappa counts as
 * a repetition without copy intent.  The copy draft is the continuation after the matched occurrence,
 * x[e*+1 ...], clipped at k and at the end of the context (§3.3 "Copy-Based Speculative Generation").
 * Returns the mode; writes draft[0..len) and *len (0 unless copy).
 */
int32_t oracle_switch(int32_t has_match, int32_t n_star, int32_t e_star, double z, float logit_tau,
                      int32_t kappa, int32_t k, const int32_t *x, int32_t L, int32_t *draft,
                      int32_t *len)
{
    int32_t mode;
    if (!has_match)
        mode = ORACLE_MODE_NO_REP;
    else if (n_star >= kappa && (float)z >= logit_tau)
        mode = ORACLE_MODE_COPY;
    else
        mode = ORACLE_MODE_REP_NO_COPY;

    *len = 0;
    if (mode == ORACLE_MODE_COPY) {
        int32_t avail = L - 1 - e_star;
        int32_t n = avail < k ? avail : k;
        for (int32_t i = 0; i < n; ++i) draft[i] = x[e_star + 1 + i];
        *len = n;
    }
    return mode;
}

/*
 * Greedy verification and append (§3.3 "Parallel Verification", "Overall Framework"; temperature 0 as
 * in the main experiments, App. A).  target has len+1 meaningful entries: the target model's argmax
 * after each draft prefix.  a = number of leading draft tokens equal to the target's argmax; the
 * context receives draft[0..a) and then target[a], the target's own next token.  If that does not fit
 * in cap the row is left untouched, *accept = -1 and the row status is ORACLE_ROW_CAPACITY.
 */
int32_t oracle_verify_row(int32_t *row, int32_t *L, int32_t cap, const int32_t *draft, int32_t len,
                          const int32_t *target, int32_t *accept)
{
    int32_t a = 0;
    while (a < len && draft[a] == target[a]) ++a;
    if (*L + a + 1 > cap) {
        *accept = -1;
        return ORACLE_ROW_CAPACITY;
    }
    for (int32_t i = 0; i < a; ++i) row[*L + i] = draft[i];
    row[*L + a] = target[a];
    *L += a + 1;
    *accept = a;
    return ORACLE_ROW_OK;
}

/*
 * One controller step over rows [b0, b1) of a batch: search, probe, switch, draft.  Layouts are the
 * documented ABI layouts: ctx [B, cap] int32, hidden [B, d] bf16, out_draft [B, k].  probe_kind 0 uses
 * probe_w = w[d]; probe_kind 1 uses probe_w = W1[H1, d] followed by w2[H1].  kappa <= 0 means
 * kappa = n_min.  out_score receives the double logit; out_n / out_e the match (0 / -1 if none).
 */
void oracle_step_rows(const int32_t *ctx, const int32_t *lens, int32_t b0, int32_t b1, int32_t cap,
                      const uint16_t *hidden, int32_t d, const uint16_t *probe_w, int32_t probe_kind,
                      int32_t H1, const float *b1v, float b2, int32_t k, int32_t n_min, int32_t n_max,
                      int32_t kappa, float logit_tau, int32_t *out_draft, int32_t *out_len,
                      int32_t *out_mode, double *out_score, int32_t *out_n, int32_t *out_e)
{
    if (kappa <= 0) kappa = n_min;
    for (int32_t b = b0; b < b1; ++b) {
        const int32_t *x = ctx + (int64_t)b * cap;
        int32_t L = lens[b];
        int32_t n_star, e_star;
        int32_t hit = oracle_longest_suffix_match(x, L, n_min, n_max, &n_star, &e_star);
        const uint16_t *h = hidden + (int64_t)b * d;
        double z;
        if (probe_kind == 0)
            z = oracle_probe_linear(h, probe_w, d);
        else
            z = oracle_probe_mlp(h, probe_w, b1v, probe_w + (int64_t)H1 * d, b2, d, H1);
        out_mode[b] = oracle_switch(hit, n_star, e_star, z, logit_tau, kappa, k, x, L,
                                    out_draft + (int64_t)b * k, &out_len[b]);
        out_score[b] = z;
        out_n[b] = n_star;
        out_e[b] = e_star;
    }
}

/* Verification over rows [b0, b1): draft [B, k], draft_len [B], target [B, k+1]. */
void oracle_verify_rows(int32_t *ctx, int32_t *lens, int32_t b0, int32_t b1, int32_t cap, int32_t k,
                        const int32_t *draft, const int32_t *draft_len, const int32_t *target,
                        int32_t *out_accept, int32_t *status)
{
    for (int32_t b = b0; b < b1; ++b) {
        int32_t st = oracle_verify_row(ctx + (int64_t)b * cap, &lens[b], cap, draft + (int64_t)b * k,
                                       draft_len[b], target + (int64_t)b * (k + 1), &out_accept[b]);
        if (status != NULL) status[b] = st;
    }
}

/*
 * Verification at temperature T > 0 (App. A runs SwitchSD with sampling; the acceptance rule is the
 * speculative-sampling rule of the works §2 builds on).  Draft token i was proposed with drafter
 * probability q[i] (q == NULL: a copy draft, which is deterministic, so q = 1) and has target
 * probability p[i] at its position.  It is accepted iff u[i] * q[i] < p[i] -- the event
 * u < min(1, p/q) for u uniform in [0, 1) -- with the product rounded to binary32 and compared in
 * binary32 (the kernel's precision; float arithmetic here is binary32).  The first rejection, at a,
 * ends the block: the appended token there is resample[a], the caller's draw from the residual
 * distribution max(0, p - q) renormalised; after len acceptances resample[len] is the bonus draw from
 * the target.  The append and the capacity rule are those of oracle_verify_row.
 */
int32_t oracle_verify_sampled_row(int32_t *row, int32_t *L, int32_t cap, const int32_t *draft, int32_t len,
                                  const float *p, const float *q, const float *u, const int32_t *resample,
                                  int32_t *accept)
{
    int32_t a = 0;
    while (a < len) {
        float qa = (q != NULL) ? q[a] : 1.0f;
        float prod = u[a] * qa;
        if (!(prod < p[a])) break;
        ++a;
    }
    if (*L + a + 1 > cap) {
        *accept = -1;
        return ORACLE_ROW_CAPACITY;
    }
    for (int32_t i = 0; i < a; ++i) row[*L + i] = draft[i];
    row[*L + a] = resample[a];
    *L += a + 1;
    *accept = a;
    return ORACLE_ROW_OK;
}

void oracle_verify_sampled_rows(int32_t *ctx, int32_t *lens, int32_t b0, int32_t b1, int32_t cap, int32_t k,
                                const int32_t *draft, const int32_t *draft_len, const float *p, const float *q,
                                const float *u, const int32_t *resample, int32_t *out_accept, int32_t *status)
{
    for (int32_t b = b0; b < b1; ++b) {
        int32_t st = oracle_verify_sampled_row(ctx + (int64_t)b * cap, &lens[b], cap, draft + (int64_t)b * k,
                                               draft_len[b], p + (int64_t)b * k,
                                               q != NULL ? q + (int64_t)b * k : NULL, u + (int64_t)b * k,
                                               resample + (int64_t)b * (k + 1), &out_accept[b]);
        if (status != NULL) status[b] = st;
    }
}

/*
 * Copy-mode label of a position (§3.2, "Problem Formulation"): position j is a copy-mode instance
 * (Y = 1) when it belongs to a verbatim sequence of at least n_train tokens that appears earlier in the
 * context (the paper sets n_train = 5).  Read as: some window x[s .. s+n-1] with s <= j <= s+n-1 also
 * occurs starting at an earlier position s' < s (the two occurrences may overlap, as in the search).
 * A longer verbatim sequence contains such a window around every one of its positions, so windows of
 * exactly n cover the definition.
 *
 * oracle_window_repeats: whether the window starting at s has an earlier occurrence (0 when the window
 * does not fit).  oracle_copy_labels: y[j] for every j < L, by the definition above, O(L^2 n).
 */
int32_t oracle_window_repeats(const int32_t *x, int32_t L, int32_t n, int32_t s)
{
    if (n < 1 || s < 0 || s + n > L) return 0;
    for (int32_t s2 = 0; s2 < s; ++s2) {
        int32_t i = 0;
        while (i < n && x[s2 + i] == x[s + i]) ++i;
        if (i == n) return 1;
    }
    return 0;
}

void oracle_copy_labels(const int32_t *x, int32_t L, int32_t n, uint8_t *y)
{
    for (int32_t j = 0; j < L; ++j) y[j] = 0;
    for (int32_t s = 0; s + n <= L; ++s)
        if (oracle_window_repeats(x, L, n, s))
            for (int32_t j = s; j < s + n; ++j) y[j] = 1;
}

/*
 * Copy candidates, W of them (§3.3 "Copy-Based Speculative Generation": up to W candidate continuations
 * of length D retrieved from the context and ranked by recency; App. D uses W = 10, D = 20).  Reading:
 * the candidates are the W most recent ends e <= L-2 at which the kappa-gram ending at the current
 * token also ends -- the common suffix of x[..e] and x[..L-1] is at least kappa tokens long (the gate
 * of the decision rule) -- listed from the most recent; candidate w continues with
 * x[e_w+1 .. e_w+len_w], len_w = min(D, L-1-e_w).  The mode follows the decision rule as in
 * oracle_switch: no repetition when no n_min-gram of the suffix occurs earlier, copy when a candidate
 * exists and the logit reaches logit_tau (compared in binary32), repetition without copy otherwise.
 * Candidates are written only for a copy row (ncand = 0 otherwise).  Returns the mode.
 */
int32_t oracle_candidates(const int32_t *x, int32_t L, int32_t n_min, int32_t n_max, int32_t kappa, double z,
                          float logit_tau, int32_t W, int32_t D, int32_t *cand, int32_t *cand_len, int32_t *ncand,
                          int32_t *cand_end)
{
    int32_t has_match = 0, n = 0;
    for (int32_t e = L - 2; e >= 0; --e) {
        /* common suffix of x[..e] and x[..L-1], at most n_max tokens */
        int32_t m = 0;
        while (m < n_max && m <= e && x[e - m] == x[L - 1 - m]) ++m;
        if (m >= n_min) has_match = 1;
        if (m >= kappa && n < W) cand_end[n++] = e;
    }
    *ncand = 0;
    if (!has_match) return ORACLE_MODE_NO_REP;
    if (n == 0 || !((float)z >= logit_tau)) return ORACLE_MODE_REP_NO_COPY;
    for (int32_t w = 0; w < n; ++w) {
        int32_t avail = L - 1 - cand_end[w];
        int32_t len = avail < D ? avail : D;
        cand_len[w] = len;
        for (int32_t i = 0; i < len; ++i) cand[(int64_t)w * D + i] = x[cand_end[w] + 1 + i];
    }
    *ncand = n;
    return ORACLE_MODE_COPY;
}

/*
 * Verification of W candidates (§3.3 "Parallel Verification with Block-Triangular Attention": the
 * target checks every candidate in one pass and the longest validated continuation is kept).  target
 * holds, per candidate w, the target's greedy token after each prefix of candidate w (D + 1 entries).
 * a_w = the leading tokens of candidate w equal to target[w]; the kept candidate is the one with the
 * largest a_w, the most recent (lowest w) on a tie; its a tokens and then target[w][a] are appended.
 * ncand = 0 counts as one empty candidate (only target[0][0] is appended).  Capacity as
 * oracle_verify_row.
 */
int32_t oracle_verify_candidates_row(int32_t *row, int32_t *L, int32_t cap, const int32_t *cand,
                                     const int32_t *cand_len, int32_t ncand, int32_t D, const int32_t *target,
                                     int32_t *accept, int32_t *choice)
{
    int32_t best = 0, a_best = -1;
    int32_t nc = ncand > 0 ? ncand : 1;
    for (int32_t w = 0; w < nc; ++w) {
        int32_t len = ncand > 0 ? cand_len[w] : 0;
        int32_t a = 0;
        while (a < len && cand[(int64_t)w * D + a] == target[(int64_t)w * (D + 1) + a]) ++a;
        if (a > a_best) {
            a_best = a;
            best = w;
        }
    }
    *choice = best;
    if (*L + a_best + 1 > cap) {
        *accept = -1;
        return ORACLE_ROW_CAPACITY;
    }
    for (int32_t i = 0; i < a_best; ++i) row[*L + i] = cand[(int64_t)best * D + i];
    row[*L + a_best] = target[(int64_t)best * (D + 1) + a_best];
    *L += a_best + 1;
    *accept = a_best;
    return ORACLE_ROW_OK;
}

/* The candidate step on rows [b0, b1): the search's match (as oracle_step_rows), the probe, and the
 * candidates and mode of oracle_candidates.  out_cand [B][W][D], out_cand_len [B][W], the rest [B]. */
void oracle_step_candidates_rows(const int32_t *ctx, const int32_t *lens, int32_t b0, int32_t b1, int32_t cap,
                                 const uint16_t *hidden, int32_t d, const uint16_t *probe_w, int32_t probe_kind,
                                 int32_t H1, const float *b1v, float b2, int32_t W, int32_t D, int32_t n_min,
                                 int32_t n_max, int32_t kappa, float logit_tau, int32_t *out_cand,
                                 int32_t *out_cand_len, int32_t *out_ncand, int32_t *out_mode, double *out_score,
                                 int32_t *out_n, int32_t *out_e, int32_t *scratch_ends)
{
    if (kappa <= 0) kappa = n_min;
    for (int32_t b = b0; b < b1; ++b) {
        const int32_t *x = ctx + (int64_t)b * cap;
        int32_t L = lens[b];
        int32_t n_star, e_star;
        oracle_longest_suffix_match(x, L, n_min, n_max, &n_star, &e_star);
        const uint16_t *h = hidden + (int64_t)b * d;
        double z;
        if (probe_kind == 0)
            z = oracle_probe_linear(h, probe_w, d);
        else
            z = oracle_probe_mlp(h, probe_w, b1v, probe_w + (int64_t)H1 * d, b2, d, H1);
        out_mode[b] = oracle_candidates(x, L, n_min, n_max, kappa, z, logit_tau, W, D,
                                        out_cand + (int64_t)b * W * D, out_cand_len + (int64_t)b * W,
                                        &out_ncand[b], scratch_ends);
        out_score[b] = z;
        out_n[b] = n_star;
        out_e[b] = e_star;
    }
}

void oracle_verify_candidates_rows(int32_t *ctx, int32_t *lens, int32_t b0, int32_t b1, int32_t cap, int32_t W,
                                   int32_t D, const int32_t *cand, const int32_t *cand_len, const int32_t *ncand,
                                   const int32_t *target, int32_t *out_accept, int32_t *out_choice, int32_t *status)
{
    for (int32_t b = b0; b < b1; ++b) {
        int32_t st = oracle_verify_candidates_row(ctx + (int64_t)b * cap, &lens[b], cap, cand + (int64_t)b * W * D,
                                                  cand_len + (int64_t)b * W, ncand[b], D,
                                                  target + (int64_t)b * W * (D + 1), &out_accept[b],
                                                  &out_choice[b]);
        if (status != NULL) status[b] = st;
    }
}
