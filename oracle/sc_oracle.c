/*
 * TEST INFRASTRUCTURE -- fp64 CPU oracle for the verification step of
 * speculative cascades (Narasimhan et al., "Faster Cascades via Speculative
 * Decoding").  Only the tests, the smoke check and the benchmark's CPU
 * baseline leg load this library; the product path never calls it.  It shares
 * no code, header or constant with the CUDA library.
 *
 * What it computes, step by step in the paper's order:
 *
 *   GenSpecSample (Algorithm 4) with the SpecCascade target (Algorithm 5):
 *     for every drafted position j < gamma of sequence b
 *       q_j = softmax(z^q_j / T), p_j = softmax(z^p_j / T)     (temperature sampling, Sec. 6)
 *       delta_j = deferral rule of Table 1:
 *          Chow: max q < 1 - alpha                              (Eq. 2)
 *          Diff: max q < max p - alpha                          (Eq. 5)
 *          OPT : max q < max p - alpha * D_TV(p, q)             (Eq. 10)
 *          with D_TV(p, q) = sum_v max(0, p(v) - q(v))          (Lemma 3)
 *       pi_j = (1 - delta_j) q_j + delta_j p_j                  (Eq. 6)
 *       a_j  = [u_{b,j} < min(1, pi_j(x_j) / q_j(x_j))]         (Algorithm 4, Bernoulli draw)
 *     a_gamma = 0;  j* = min{ j : a_j = 0 }
 *     next token ~ norm(max(0, pi_{j*} - q_{j*}))  if j* < gamma
 *                ~ pi_gamma                         otherwise
 *
 *   or with the token-specific target (Section 4.4, TokenSpecCascade):
 *       r_j(v) in {0, 1} per token by a plug-in rule:
 *          TokenV1: q(v) < max p - alpha
 *          TokenV2: p(v) < max p - alpha
 *          TokenV3: p(v) < max p * (1 - alpha)
 *       eta_j = sum_v r_j(v) q_j(v)
 *       pi_j(v) = q_j(v) (1 - r_j(v)) + eta_j p_j(v)
 *     and the same acceptance, first rejection and residual draw;
 *
 *   or the other targets of Table 3 run through Algorithm 4:
 *       Lossy speculative decoding:  pi(v) = max{ min{ q(v), p(v)/(1 - alpha) }, p(v)/beta }
 *          (Lemma 2: the acceptance is min(1, p(x)/((1 - alpha) q(x))) and the residual
 *          norm(max(0, p/beta - q)); pi need not sum to one), beta >= 1 - alpha;
 *          alpha = 1 is the limit alpha -> 1-: p(v)/(1 - alpha) is +infinity where
 *          p(v) > 0 and 0 where p(v) = 0, so a draft with p(x) = 0 is still rejected;
 *       BiLD*:  delta = 1(D(q, p) > alpha), D(q, p) = -sum_v q(v) log p(v) (the
 *          temperature-sampling discrepancy of the experiments' appendix; with
 *          greedy decoding the appendix's -log p(argmax q)),
 *          pi = (1 - delta) q + delta p;
 *
 *   or the log-loss plug-in rules (appendix on log loss), delta by entropies:
 *       ChowLog: H(q) > alpha;   DiffLog: sum q log q < sum p log p - alpha;
 *       OPTLog:  sum q log q < sum p log p - alpha D_TV(p, q);
 *
 *   and, with T = 0, greedy decoding (appendix, the greedy special case): the
 *   rule is evaluated on the untempered softmax (T = 1) except that its D_TV is
 *   that of the one-hot q~, p~ at the argmaxes (lowest index on ties), i.e.
 *   1(argmax q != argmax p), as in the greedy lemma, and BiLD*'s discrepancy is
 *   -log p(argmax q) as the experiments' appendix sets it for greedy decoding;
 *   pi = (1 - delta) q~ + delta p~,
 *   and Algorithm 4 runs on those:
 *   a draft is rejected only when delta = 1 and it is not the verifier's argmax,
 *   and the residual (and bonus) token is the verifier's argmax.
 *
 * Readings where the paper leaves a choice open:
 *   - the bonus position has no draft row, so pi_gamma := p_gamma (as in
 *     SpecDecode, Algorithm 1);
 *   - the Bernoulli draw of position j is "u_{b,j} < rho" with the supplied
 *     uniform u in [0, 1); a draft whose q(x) <= pi(x) is always accepted, and
 *     so is a draft with q(x) = 0;
 *   - the single uniform u_{b,gamma} drives the residual or bonus sample, by
 *     inverse CDF in ascending vocabulary order: the smallest k whose cumulative
 *     weight C_k exceeds u * R, R the total weight;
 *   - the deferral inequalities are strict, as printed in Table 1.
 *
 * Decision margins: for every decision that depends on a floating-point
 * comparison, the oracle records how far it was from flipping (deferral:
 * |lhs - rhs|; acceptance: |u - pi(x)/q(x)|; sample: distance of u*R to the
 * nearest cumulative boundary, relative to R).  A sequence whose smallest
 * margin over positions 0..j* is below 1e-6 is "flagged": an fp32 computation
 * may legitimately decide it the other way.
 *
 * Everything is fp64 with Neumaier-compensated sums; bf16 logits are widened
 * exactly.  One sequence per OpenMP iteration.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_F32 0
#define OR_BF16 1

#define OR_CHOW 0
#define OR_DIFF 1
#define OR_OPT 2
#define OR_ALWAYS 3 /* delta = 1: standard speculative sampling (Algorithm 1) */
#define OR_NEVER 4  /* delta = 0: pi = q */
#define OR_TOKEN_V1 5 /* token-specific: r(v) = [q(v) < max p - alpha] */
#define OR_TOKEN_V2 6 /* token-specific: r(v) = [p(v) < max p - alpha] */
#define OR_TOKEN_V3 7 /* token-specific: r(v) = [p(v) < max p (1 - alpha)] */
#define OR_LOSSY 8    /* lossy speculative decoding target (Table 3, Lemma 2), parameter beta */
#define OR_BILD 9     /* BiLD*: delta = 1(D(q, p) > alpha), D = -sum_v q(v) log p(v) (T > 0) or -log p(argmax q) (T = 0) */
#define OR_CHOW_LOG 10 /* H(q) > alpha */
#define OR_DIFF_LOG 11 /* sum q log q < sum p log p - alpha */
#define OR_OPT_LOG 12  /* sum q log q < sum p log p - alpha D_TV(p, q) */

/* per-row record layout, [B][gamma][OR_ROW_FIELDS] */
#define OR_ROW_MAXQ 0
#define OR_ROW_MAXP 1
#define OR_ROW_TV 2
#define OR_ROW_DELTA 3
#define OR_ROW_ACCEPT 4
#define OR_ROW_QX 5
#define OR_ROW_PIX 6
#define OR_ROW_MARGIN_DELTA 7
#define OR_ROW_MARGIN_ACCEPT 8
#define OR_ROW_FIELDS 9

/* per-sequence record layout, [B][OR_SEQ_FIELDS] */
#define OR_SEQ_MIN_MARGIN 0
#define OR_SEQ_SAMPLE_MARGIN 1
#define OR_SEQ_STATUS 2
#define OR_SEQ_BONUS_MAXP 3
#define OR_SEQ_FIELDS 4

/* status bits of a sequence with invalid input */
#define OR_BAD_TOKEN 1
#define OR_BAD_LOGIT 2
#define OR_BAD_UNIFORM 4

/* ------------------------------------------------------------ helpers */

static double logit_at(const void *base, int dtype, size_t i)
{
    if (dtype == OR_BF16) {
        uint32_t w = (uint32_t)((const uint16_t *)base)[i] << 16;
        float f;
        memcpy(&f, &w, sizeof f);
        return (double)f;
    }
    return (double)((const float *)base)[i];
}

/* Neumaier's compensated summation. */
typedef struct {
    double s, c;
} csum;

static void csum_add(csum *k, double x)
{
    double t = k->s + x;
    if (fabs(k->s) >= fabs(x))
        k->c += (k->s - t) + x;
    else
        k->c += (x - t) + k->s;
    k->s = t;
}

static double csum_value(const csum *k) { return k->s + k->c; }

/*
 * Tempered softmax of one row: probs[v] = exp(z_v/T - M) / S, with
 * M = max_v z_v/T and S = sum_v exp(z_v/T - M).  Returns 0, or -1 when the row
 * is not a distribution (a NaN or +inf logit, or every logit -inf).
 */
static int tempered_softmax_ln(const void *z, int dtype, size_t off, int V, double T,
                               double *probs, double *M_out, double *lnS_out)
{
    double M = -INFINITY;
    for (int v = 0; v < V; ++v) {
        double y = logit_at(z, dtype, off + (size_t)v);
        if (isnan(y) || y == INFINITY)
            return -1;
        y = y / T;
        probs[v] = y;
        if (y > M)
            M = y;
    }
    if (!isfinite(M))
        return -1;
    csum S = {0.0, 0.0};
    for (int v = 0; v < V; ++v) {
        double e = exp(probs[v] - M);
        probs[v] = e;
        csum_add(&S, e);
    }
    double s = csum_value(&S);
    for (int v = 0; v < V; ++v)
        probs[v] /= s;
    if (M_out)
        *M_out = M;
    if (lnS_out)
        *lnS_out = log(s);
    return 0;
}

static int tempered_softmax(const void *z, int dtype, size_t off, int V, double T,
                            double *probs)
{
    return tempered_softmax_ln(z, dtype, off, V, T, probs, NULL, NULL);
}

/* ln of the tempered probability of token x: z_x/T - M - ln S (no underflow). */
static double log_prob(const void *z, int dtype, size_t off, int x, double T, double M,
                       double lnS)
{
    return logit_at(z, dtype, off + (size_t)x) / T - M - lnS;
}

static double max_of(const double *x, int V)
{
    double m = x[0];
    for (int v = 1; v < V; ++v)
        if (x[v] > m)
            m = x[v];
    return m;
}

/* D_TV(p, q) = sum_v max(0, p(v) - q(v))  (Lemma 3; equals 0.5 * ||p - q||_1). */
static double tv_distance(const double *p, const double *q, int V)
{
    csum t = {0.0, 0.0};
    for (int v = 0; v < V; ++v) {
        double d = p[v] - q[v];
        if (d > 0.0)
            csum_add(&t, d);
    }
    return csum_value(&t);
}

/*
 * Deferral decision delta(q, p) of Table 1 from the three row scalars.
 * *margin receives |lhs - rhs| of the strict inequality (infinity for the two
 * constant rules).
 */
static int deferral(int rule, double alpha, double maxq, double maxp, double tv, double *margin)
{
    double lhs = maxq, rhs;
    switch (rule) {
    case OR_CHOW: rhs = 1.0 - alpha; break;        /* Eq. 2  */
    case OR_DIFF: rhs = maxp - alpha; break;       /* Eq. 5  */
    case OR_OPT: rhs = maxp - alpha * tv; break;   /* Eq. 10 */
    case OR_ALWAYS: *margin = INFINITY; return 1;
    default: *margin = INFINITY; return 0;
    }
    *margin = fabs(lhs - rhs);
    return lhs < rhs ? 1 : 0;
}

/*
 * Token-specific deferral of token v (Section 4.4): r(v) = 1 when the token is
 * deferred to the target model.  lnp_rel = ln p(v) - ln max p, formed from the
 * logits, is what TokenV3 compares (p(v) < max p (1 - alpha) <=> lnp_rel <
 * ln(1 - alpha)); TokenV1 and TokenV2 compare probabilities with max p - alpha.
 * *margin receives |lhs - rhs| in the units compared.
 */
static int token_r(int rule, double alpha, double qv, double pv, double maxp, double lnp_rel,
                   double *margin)
{
    double lhs, rhs;
    switch (rule) {
    case OR_TOKEN_V1: lhs = qv; rhs = maxp - alpha; break;
    case OR_TOKEN_V2: lhs = pv; rhs = maxp - alpha; break;
    default:
        if (alpha >= 1.0) { *margin = INFINITY; return 0; }   /* ln(0): nothing deferred */
        lhs = lnp_rel; rhs = log1p(-alpha);
        if (alpha == 0.0 && lnp_rel == 0.0) { *margin = INFINITY; return 0; }  /* the mode itself, exactly */
        break;
    }
    *margin = fabs(lhs - rhs);
    return lhs < rhs ? 1 : 0;
}

/*
 * The token-specific target of one row: r(v) for every token, eta = sum_v r(v) q(v)
 * and pi(v) = q(v) (1 - r(v)) + eta p(v).  r is written to rv[] (0/1); the
 * returned margin is the smallest per-token margin among tokens with q(v) or
 * p(v) of at least 1e-9 (flipping a lighter token moves eta and pi by less),
 * and always includes that of the draft token x (x < 0: none), whose own r(x)
 * decides whether it is kept outright, whatever its mass.
 */
static double token_target(int rule, double alpha, const void *zp, int dtype, size_t poff, double Mp,
                           double T, const double *q, const double *p, int V, double maxp, int x,
                           double *rv, double *pi, double *margin)
{
    csum eta = {0.0, 0.0};
    double mmin = INFINITY;
    for (int v = 0; v < V; ++v) {
        double m;
        const double lnp_rel = logit_at(zp, dtype, poff + v) / T - Mp;  /* as the softmax forms y / T */
        const int r = token_r(rule, alpha, q[v], p[v], maxp, lnp_rel, &m);
        rv[v] = r;
        if (r) csum_add(&eta, q[v]);
        if ((q[v] >= 1e-9 || p[v] >= 1e-9 || v == x) && m < mmin) mmin = m;
    }
    const double e = csum_value(&eta);
    if (pi)
        for (int v = 0; v < V; ++v)
            pi[v] = q[v] * (1.0 - rv[v]) + e * p[v];
    *margin = mmin;
    return e;
}

/* sum_v x(v) log x(v) of a distribution (0 log 0 = 0): minus its entropy. */
static double neg_entropy(const double *x, int V)
{
    csum s = {0.0, 0.0};
    for (int v = 0; v < V; ++v)
        if (x[v] > 0.0)
            csum_add(&s, x[v] * log(x[v]));
    return csum_value(&s);
}

/* Lowest index of the largest entry. */
static int argmax_of(const double *x, int V)
{
    int a = 0;
    for (int v = 1; v < V; ++v)
        if (x[v] > x[a])
            a = v;
    return a;
}

/* The lossy speculative-decoding target of one token (Table 3). */
static double lossy_pi(double qv, double pv, double alpha, double beta)
{
    double a = alpha < 1.0 ? pv / (1.0 - alpha) : (pv > 0.0 ? INFINITY : 0.0);  /* alpha -> 1- */
    double m = qv < a ? qv : a;
    double b = pv / beta;
    return m > b ? m : b;
}

/*
 * BiLD*'s discrepancy D(q, p) = -sum_v q(v) log p(v) of one row pair, with
 * log p(v) from the logits.  It is +infinity when some q(v) > 0 has p(v) = 0:
 * q(v) > 0 exactly when the draft logit is finite (whether or not exp of it
 * underflows in fp64), p(v) = 0 exactly when the target logit is -infinity.
 */
static double cross_entropy(const double *q, const void *zq, size_t qoff, const void *zp, int dtype,
                            size_t poff, int V, double T, double Mp, double lnSp)
{
    csum D = {0.0, 0.0};
    for (int v = 0; v < V; ++v) {
        if (!(logit_at(zq, dtype, qoff + (size_t)v) > -INFINITY))
            continue;  /* q(v) = 0 */
        const double lp = log_prob(zp, dtype, poff, v, T, Mp, lnSp);
        if (lp == -INFINITY)
            return INFINITY;
        if (q[v] > 0.0)
            csum_add(&D, -q[v] * lp);
    }
    return csum_value(&D);
}

/*
 * Inverse-CDF draw from the unnormalised weights w[0..V-1] >= 0 with the
 * uniform u: the smallest k with C_k = sum_{v<=k} w_v > u * R, R = sum_v w_v.
 * If rounding leaves u*R at or above the last cumulative value, the largest k
 * with w_k > 0 is taken.  *margin = min(u R - C_{k-1}, C_k - u R) / R.
 * Returns -1 when R == 0.
 */
static int inverse_cdf(const double *w, int V, double u, double *margin)
{
    csum R = {0.0, 0.0};
    for (int v = 0; v < V; ++v)
        csum_add(&R, w[v]);
    double r = csum_value(&R);
    if (!(r > 0.0)) {
        *margin = 0.0;
        return -1;
    }
    double t = u * r;
    csum C = {0.0, 0.0};
    double prev = 0.0;
    for (int k = 0; k < V; ++k) {
        csum_add(&C, w[k]);
        double c = csum_value(&C);
        if (c > t) {
            double m1 = t - prev, m2 = c - t;
            *margin = (m1 < m2 ? m1 : m2) / r;
            return k;
        }
        prev = c;
    }
    *margin = 0.0;
    for (int k = V - 1; k >= 0; --k)
        if (w[k] > 0.0)
            return k;
    return -1;
}

/* ------------------------------------------------------------ one sequence */

static void verify_sequence(const void *draft, const void *target, int dtype,
                            const int32_t *tokens, const float *uniforms, int b, int gamma,
                            int V, int rule, double alpha, double beta, double T, int32_t *num_accepted,
                            int32_t *next_token, double *row_info, double *seq_info,
                            double *q, double *p, double *w)
{
    const size_t dbase = (size_t)b * gamma * V;
    const size_t tbase = (size_t)b * (gamma + 1) * V;
    const int32_t *x = tokens + (size_t)b * gamma;
    const float *u = uniforms + (size_t)b * (gamma + 1);
    int status = 0;
    for (int j = 0; j < gamma; ++j)
        if (x[j] < 0 || x[j] >= V)
            status |= OR_BAD_TOKEN;
    for (int j = 0; j <= gamma; ++j)
        if (!(u[j] >= 0.0f && u[j] < 1.0f))
            status |= OR_BAD_UNIFORM;

    const int greedy = !(T > 0.0);       /* T = 0: greedy decoding */
    const double Tr = greedy ? 1.0 : T;   /* temperature of the rule's distributions */
    const int token = rule >= OR_TOKEN_V1 && rule <= OR_TOKEN_V3;
    const int lossy = rule == OR_LOSSY;
    int jstar = gamma;          /* a_gamma = 0 */
    double min_margin = INFINITY;
    int delta_star = 0;         /* delta at j* */
    for (int j = 0; j < gamma; ++j) {
        double Mq, lnSq, Mp, lnSp;
        int okq = tempered_softmax_ln(draft, dtype, dbase + (size_t)j * V, V, Tr, q, &Mq, &lnSq);
        int okp = tempered_softmax_ln(target, dtype, tbase + (size_t)j * V, V, Tr, p, &Mp, &lnSp);
        if (okq || okp) {
            status |= OR_BAD_LOGIT;
            continue;
        }
        double maxq = max_of(q, V), maxp = max_of(p, V), tv = tv_distance(p, q, V);
        if (greedy)  /* the rules' D_TV is that of the one-hot q~, p~: 1(argmax q != argmax p) */
            tv = argmax_of(q, V) != argmax_of(p, V);
        double m_delta, m_acc = INFINITY;
        int delta;
        int accept = 1;
        double qx = 0.0, pix = 0.0;
        if (token) {
            /* token-specific target (TokenSpecCascade): w holds r(v) for this row */
            const double eta = token_target(rule, alpha, target, dtype, tbase + (size_t)j * V, Mp, Tr,
                                            q, p, V, maxp, (status & OR_BAD_TOKEN) ? -1 : x[j], w, NULL,
                                            &m_delta);
            delta = 0;
            if (!(status & OR_BAD_TOKEN)) {
                const int rx = (int)w[x[j]];
                delta = rx; /* reported: r(x_j), the draft token's own deferral */
                qx = q[x[j]];
                pix = qx * (1 - rx) + eta * p[x[j]];
                if (rx) {
                    /* pi(x)/q(x) = eta p(x)/q(x), from log-probabilities; a draft with
                       q(x) <= pi(x) (or q(x) = 0) is always accepted */
                    double lq = log_prob(draft, dtype, dbase + (size_t)j * V, x[j], Tr, Mq, lnSq);
                    double lp = log_prob(target, dtype, tbase + (size_t)j * V, x[j], Tr, Mp, lnSp);
                    double ratio = eta > 0.0 ? exp(lp - lq + log(eta)) : 0.0;
                    if (lq > -INFINITY && ratio < 1.0) {
                        accept = (double)u[j] < ratio;
                        m_acc = fabs((double)u[j] - ratio);
                    }
                }
            }
        } else if (lossy) {
            /* pi(x)/q(x) = max{ min{1, (p/q)/(1 - alpha)}, (p/q)/beta }, from log-probabilities */
            delta = 1;
            m_delta = INFINITY;
            if (!(status & OR_BAD_TOKEN)) {
                qx = q[x[j]];
                pix = lossy_pi(qx, p[x[j]], alpha, beta);
                double lq = log_prob(draft, dtype, dbase + (size_t)j * V, x[j], Tr, Mq, lnSq);
                double lp = log_prob(target, dtype, tbase + (size_t)j * V, x[j], Tr, Mp, lnSp);
                if (lq > -INFINITY) {
                    double pq = exp(lp - lq);
                    double a = alpha < 1.0 ? pq / (1.0 - alpha) : (pq > 0.0 ? INFINITY : 0.0);
                    double ratio = a < 1.0 ? a : 1.0;
                    if (pq / beta > ratio) ratio = pq / beta;
                    if (ratio < 1.0) {
                        accept = (double)u[j] < ratio;
                        m_acc = fabs((double)u[j] - ratio);
                    }
                }
            }
        } else if (rule >= OR_CHOW_LOG) {
            const double nhq = neg_entropy(q, V), nhp = neg_entropy(p, V);
            double lhs = nhq, rhs;
            if (rule == OR_CHOW_LOG) { lhs = -nhq; rhs = alpha; delta = lhs > rhs; }  /* H(q) > alpha */
            else {
                rhs = rule == OR_DIFF_LOG ? nhp - alpha : nhp - alpha * tv;
                delta = lhs < rhs;
            }
            m_delta = fabs(lhs - rhs);
        } else if (rule == OR_BILD) {
            /* greedy decoding: the BiLD baseline's D(q, p) = -log p(argmax q); with a
               temperature, its analogue -sum_v q(v) log p(v) */
            const double D = greedy ? -log_prob(target, dtype, tbase + (size_t)j * V, argmax_of(q, V), Tr, Mp, lnSp)
                                    : cross_entropy(q, draft, dbase + (size_t)j * V, target, dtype,
                                                    tbase + (size_t)j * V, V, Tr, Mp, lnSp);
            delta = D > alpha;  /* strict, as printed */
            m_delta = isfinite(D) ? fabs(D - alpha) : INFINITY;
        } else {
            delta = deferral(rule, alpha, maxq, maxp, tv, &m_delta);
        }
        if (greedy && !(status & OR_BAD_TOKEN)) {
            /* one-hot q~, p~: pi(x)/q~(x) is 1 unless delta = 1 and x is not p's
               argmax (then 0); a draft with q~(x) = 0 is accepted (reading 3) */
            const int aq = argmax_of(q, V), ap = argmax_of(p, V);
            qx = x[j] == aq;
            pix = delta ? (double)(x[j] == ap) : qx;
            accept = !(qx && delta && x[j] != ap);
        } else if (!token && !lossy && !(status & OR_BAD_TOKEN)) {
            qx = q[x[j]];
            pix = delta ? p[x[j]] : qx; /* pi(x) = (1 - delta) q(x) + delta p(x) */
            if (delta) {
                /* pi(x)/q(x) = p(x)/q(x), formed from log-probabilities so that it
                   stays exact when both underflow; q(x) <= pi(x) always accepts
                   (q(x) = 0 only for a -inf logit) */
                double lq = log_prob(draft, dtype, dbase + (size_t)j * V, x[j], Tr, Mq, lnSq);
                double lp = log_prob(target, dtype, tbase + (size_t)j * V, x[j], Tr, Mp, lnSp);
                if (lq > lp) {
                    double ratio = exp(lp - lq);
                    accept = (double)u[j] < ratio;
                    m_acc = fabs((double)u[j] - ratio);
                }
            }
        }
        if (row_info) {
            double *r = row_info + ((size_t)b * gamma + j) * OR_ROW_FIELDS;
            r[OR_ROW_MAXQ] = maxq;
            r[OR_ROW_MAXP] = maxp;
            r[OR_ROW_TV] = tv;
            r[OR_ROW_DELTA] = delta;
            r[OR_ROW_ACCEPT] = accept;
            r[OR_ROW_QX] = qx;
            r[OR_ROW_PIX] = pix;
            r[OR_ROW_MARGIN_DELTA] = m_delta;
            r[OR_ROW_MARGIN_ACCEPT] = m_acc;
        }
        if (j <= jstar) {
            if (m_delta < min_margin) min_margin = m_delta;
            if (m_acc < min_margin) min_margin = m_acc;
        }
        if (!accept && j < jstar) {
            jstar = j;
            delta_star = delta;
        }
    }

    /* The bonus row is always checked, so that its max p is reported. */
    double bonus_maxp = NAN;
    if (tempered_softmax(target, dtype, tbase + (size_t)gamma * V, V, Tr, p) == 0)
        bonus_maxp = max_of(p, V);
    else
        status |= OR_BAD_LOGIT;

    int tok = -1;
    double m_sample = 0.0;
    if (status == 0 && greedy) {
        /* the residual max(0, pi - q~) = delta max(0, p~ - q~) of row j*, and the
           bonus pi_gamma = p~_gamma, are one-hot at the verifier's argmax */
        tempered_softmax(target, dtype, tbase + (size_t)jstar * V, V, Tr, p);
        tok = argmax_of(p, V);
        m_sample = INFINITY;
        num_accepted[b] = jstar;
        next_token[b] = tok;
    } else if (status == 0) {
        if (jstar < gamma && token) {
            /* residual norm(max(0, pi - q)) of row j* with the token-specific
               target: max(0, eta p(v) - r(v) q(v)) */
            double Mp, lnSp, m_unused;
            tempered_softmax(draft, dtype, dbase + (size_t)jstar * V, V, Tr, q);
            tempered_softmax_ln(target, dtype, tbase + (size_t)jstar * V, V, Tr, p, &Mp, &lnSp);
            const double eta = token_target(rule, alpha, target, dtype, tbase + (size_t)jstar * V, Mp,
                                            Tr, q, p, V, max_of(p, V), -1, w, NULL, &m_unused);
            for (int v = 0; v < V; ++v) {
                double d = eta * p[v] - w[v] * q[v];
                w[v] = d > 0.0 ? d : 0.0;
            }
            tok = inverse_cdf(w, V, (double)u[gamma], &m_sample);
        } else if (jstar < gamma && lossy) {
            /* residual norm(max(0, pi - q)) of row j* with the lossy target */
            tempered_softmax(draft, dtype, dbase + (size_t)jstar * V, V, Tr, q);
            tempered_softmax(target, dtype, tbase + (size_t)jstar * V, V, Tr, p);
            for (int v = 0; v < V; ++v) {
                double d = lossy_pi(q[v], p[v], alpha, beta) - q[v];
                w[v] = d > 0.0 ? d : 0.0;
            }
            tok = inverse_cdf(w, V, (double)u[gamma], &m_sample);
        } else if (jstar < gamma) {
            /* residual norm(max(0, pi - q)) of row j*; pi = p there since a
               rejection implies delta = 1 */
            tempered_softmax(draft, dtype, dbase + (size_t)jstar * V, V, Tr, q);
            tempered_softmax(target, dtype, tbase + (size_t)jstar * V, V, Tr, p);
            for (int v = 0; v < V; ++v) {
                double pi = delta_star ? p[v] : q[v];
                double d = pi - q[v];
                w[v] = d > 0.0 ? d : 0.0;
            }
            tok = inverse_cdf(w, V, (double)u[gamma], &m_sample);
        } else {
            /* bonus position: sample from pi_gamma = p_gamma (p still holds it) */
            tok = inverse_cdf(p, V, (double)u[gamma], &m_sample);
        }
        if (m_sample < min_margin)
            min_margin = m_sample;
        num_accepted[b] = jstar;
        next_token[b] = tok;
    } else {
        num_accepted[b] = 0;
        next_token[b] = -1;
        min_margin = 0.0;
    }
    if (seq_info) {
        double *s = seq_info + (size_t)b * OR_SEQ_FIELDS;
        s[OR_SEQ_MIN_MARGIN] = min_margin;
        s[OR_SEQ_SAMPLE_MARGIN] = m_sample;
        s[OR_SEQ_STATUS] = status;
        s[OR_SEQ_BONUS_MAXP] = bonus_maxp;
    }
}

/* ------------------------------------------------------------ exported API */

int oracle_row_fields(void) { return OR_ROW_FIELDS; }
int oracle_seq_fields(void) { return OR_SEQ_FIELDS; }

int oracle_num_threads(int nthreads)
{
#ifdef _OPENMP
    return nthreads > 0 ? nthreads : omp_get_max_threads();
#else
    (void)nthreads;
    return 1;
#endif
}

/*
 * The whole verification step for B sequences.
 *   draft    [B][gamma][V]   f32 or bf16 bits (dtype)
 *   target   [B][gamma+1][V]
 *   tokens   [B][gamma] int32,   uniforms [B][gamma+1] float32
 *   num_accepted, next_token   [B] outputs (0 and -1 for an invalid sequence)
 *   row_info [B][gamma][OR_ROW_FIELDS] or NULL;  seq_info [B][OR_SEQ_FIELDS] or NULL
 * Returns 0, or -1 on bad arguments.
 */
int oracle_verify(const void *draft, const void *target, int dtype, const int32_t *tokens,
                  const float *uniforms, int B, int gamma, int V, int rule, double alpha,
                  double beta, double T, int32_t *num_accepted, int32_t *next_token,
                  double *row_info, double *seq_info, int nthreads)
{
    if (!draft || !target || !tokens || !uniforms || !num_accepted || !next_token)
        return -1;
    if (B < 0 || gamma < 1 || V < 1 || !(T >= 0.0) || rule < 0 || rule > OR_OPT_LOG)
        return -1;
    if (T == 0.0 && ((rule >= OR_TOKEN_V1 && rule <= OR_TOKEN_V3) || rule == OR_LOSSY))
        return -1;  /* greedy decoding is defined for the scalar deferral rules */
    if (rule == OR_LOSSY && !(beta > 0.0 && beta >= 1.0 - alpha))
        return -1;
    int failed = 0;
#ifdef _OPENMP
#pragma omp parallel num_threads(oracle_num_threads(nthreads)) reduction(| : failed)
#endif
    {
        double *q = malloc(sizeof(double) * (size_t)V);
        double *p = malloc(sizeof(double) * (size_t)V);
        double *w = malloc(sizeof(double) * (size_t)V);
        if (!q || !p || !w) {
            failed = 1;
        } else {
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
            for (int b = 0; b < B; ++b)
                verify_sequence(draft, target, dtype, tokens, uniforms, b, gamma, V, rule, alpha,
                                beta, T, num_accepted, next_token, row_info, seq_info, q, p, w);
        }
        free(q);
        free(p);
        free(w);
    }
    return failed ? -1 : 0;
}

/*
 * Per-pair statistics (max q, max p, D_TV) for every (b, j < gamma):
 * outputs [B*gamma].  Returns 0, or -1 (bad arguments or an invalid row).
 */
int oracle_row_stats(const void *draft, const void *target, int dtype, int B, int gamma, int V,
                     double T, double *maxq, double *maxp, double *tv, int nthreads)
{
    if (!draft || !target || !maxq || !maxp || !tv || B < 0 || gamma < 1 || V < 1 || !(T > 0.0))
        return -1;
    int bad = 0;
#ifdef _OPENMP
#pragma omp parallel num_threads(oracle_num_threads(nthreads)) reduction(| : bad)
#endif
    {
        double *q = malloc(sizeof(double) * (size_t)V);
        double *p = malloc(sizeof(double) * (size_t)V);
        if (!q || !p) {
            bad = 1;
        } else {
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
            for (int r = 0; r < B * gamma; ++r) {
                int b = r / gamma, j = r % gamma;
                int e1 = tempered_softmax(draft, dtype, (size_t)r * V, V, T, q);
                int e2 = tempered_softmax(target, dtype, ((size_t)b * (gamma + 1) + j) * V, V, T, p);
                if (e1 || e2) {
                    bad = 1;
                    maxq[r] = maxp[r] = tv[r] = NAN;
                    continue;
                }
                maxq[r] = max_of(q, V);
                maxp[r] = max_of(p, V);
                tv[r] = tv_distance(p, q, V);
            }
        }
        free(q);
        free(p);
    }
    return bad ? -1 : 0;
}

/* Exported building blocks, for pinning each step on its own. */
int oracle_softmax(const void *z, int dtype, int V, double T, double *probs)
{
    if (!z || !probs || V < 1 || !(T > 0.0))
        return -1;
    return tempered_softmax(z, dtype, 0, V, T, probs);
}

double oracle_tv(const double *p, const double *q, int V) { return tv_distance(p, q, V); }

int oracle_deferral(int rule, double alpha, double maxq, double maxp, double tv, double *margin)
{
    double m;
    int d = deferral(rule, alpha, maxq, maxp, tv, &m);
    if (margin)
        *margin = m;
    return d;
}

int oracle_inverse_cdf(const double *w, int V, double u, double *margin)
{
    double m;
    int k = inverse_cdf(w, V, u, &m);
    if (margin)
        *margin = m;
    return k;
}
