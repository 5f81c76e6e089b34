/*
 * vsd_oracle.c -- plain CPU oracle for the E-step / M-step of Variational
 * Speculative Decoding (VSD), arxiv 2602.05774.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * statement of what the GPU path must compute.  Only the test suite, the
 * smoke check and the benchmark's CPU-baseline leg may load it.  It shares no
 * code, header, table or helper with the CUDA library, and it includes nothing
 * from it.
 *
 * Arithmetic: IEEE double throughout, sequential summation over v ascending,
 * inputs read as the exact float values they hold (bf16 inputs arrive widened
 * to float, which is exact).  Build without -ffast-math.
 *
 * Notation (paper, Table 7 and Algorithm 1):
 *   prefix x  -> index b (0..B-1)
 *   proposal s = 1..S  -> index s (0..K-1), K plays the paper's S
 *   length l = 1..L    -> depth index d (0..D-1), l = d+1, D plays the paper's L
 *   q = q_psi (draft), p = p_theta (target), both at temperature T (Eq. 1).
 * Logit rows are [B][K][D][V], row r = (b*K + s)*D + d, V contiguous.
 *
 * Readings of the paper taken here (each is listed in the design notes):
 *   R1  Proposals are K nested paths of depth D: z~^{(s)}_{<=l} is the first l
 *       tokens of path s (Algorithm 1 draws one proposal per (l,s); nested
 *       prefixes of one depth-D path have the same per-l marginal).
 *   R2  The row (s,d) is the caller's distribution conditioned on
 *       (x, z~^{(s)}_{<d}) (teacher forcing); the oracle never re-conditions.
 *   R3  The substitute path z' of Algorithm 1 is the speculative correction of
 *       Sec. 3: accepted prefix, then a residual token norm(max(0,p-q)) at the
 *       first rejection, then p-samples from the given rows.
 *   R4  The greedy reference z-bar of Algorithm 2 is taken per path from the
 *       same rows: v-bar_d = argmax p_{s,d} (lowest index on ties), unless the
 *       caller passes ref_logkappa[b][l].
 *   R5  o~ is the binary validity I[log k(z~) >= log k(z-bar)]; o' carries
 *       w(l) = w_base^l (Sec. 4.3 text next to Eq. beta; App. F w(l)=1.05^l).
 *   R6  beta with an empty or zero leave-one-out denominator is 0.
 *   R7  zeta is the softmax over all K proposals of q(z~_{<=l})/tau (literal
 *       reading: a path probability); zeta_mode=1 uses log q(z~_{<=l}).
 *   R8  loss_b = -J_b / N_b (0 if N_b = 0), reported loss = mean over b;
 *       beta, zeta, o~, o', N_b are constants of the gradient (Eq. advance).
 *   R9  Ties: accept on u <= alpha (Eq. 1 text "r <= alpha"); sample = smallest
 *       v with u < F(v); argmax lowest index; ">=" passes in Algorithm 2.
 *   R10 If the residual mass sum_v max(0,p-q) is 0 the correction samples p.
 *   R11 VSD (KL): the KL term of the ELBO (Eq. elbo_vi) is replaced by the
 *       top-K renormalised cross-entropy of Eq. klv (K = 10) at every row the
 *       proposals visit; per prefix L_KL = (1/S) sum_{s,d} L_topK(row (s,d)),
 *       an MC estimate of the path-level KL, which is a sum over positions;
 *       loss_b = -J_b/N_b + kl_weight L_KL.  The paper gives no weight;
 *       kl_weight = 0 is VSD without the term.  The rows' contexts are held
 *       fixed in the gradient (as in R8).
 *   R12 T = 0 (greedy decoding, the T in {0, 1} of the paper's tables): every
 *       decision takes the T -> 0 limit of Eq. 1's distributions, q and p
 *       one-hot at their argmax (lowest index on ties): z~ = argmax q,
 *       alpha = [argmax p = z~], the residual and the later samples are
 *       argmax p.  The M-step's log-likelihood (Eq. advance), zeta and the
 *       top-K term use the draft's distribution at temperature 1, since log q
 *       at T = 0 is not finite.
 *   R14 Tree verification with the sequential sibling rule (lossless
 *       multi-draft; App. E trees): at a node on the accepted path its
 *       children are tried in node order; child i is accepted with
 *       probability min(1, p_i(t_i)/q_i(t_i)), where p_1 = p, q_1 = q,
 *       p_{i+1} = norm(max(0, p_i - q_i)) (p_i kept if that has no mass) and
 *       q_{i+1} = q_i with t_i removed and renormalised (siblings are distinct
 *       draws, as without replacement); the first accepted child continues
 *       the path and later siblings are not tried; if every child is
 *       rejected, the correction token is drawn from p_{m+1} with the last
 *       child's uniform.  Output is distributed as p whenever t_i ~ q_i.
 *   R15 Tree EM (App. E trees as latent proposals): every node n >= 1 is the
 *       proposal z~(n) = the tokens on its root path, of length l = depth(n).
 *       Each position x on a path is verified alone as in R3 (independent
 *       rule, the path validity of Eq. 2): z'_x = t_x on an accepted path, the
 *       residual at the first rejected node, p-draws below it (with each
 *       node's own u_correct); the reference per row is R4's argmax.  o~, o'
 *       as R5 with w(depth); beta and zeta are taken over the nodes of one
 *       depth (the proposals of one length); loss and gradient as Eq.
 *       advance, each node's row collecting the terms of every proposal
 *       whose path goes through one of its children.
 *   R13 A greedy reference path supplied as rows (Algorithm 2's z-bar drawn
 *       from the greedy target policy, with the draft and target rows along
 *       it): log k(z-bar_{<=l}) = sum_{d<=l} log min(1, p_d(v_d)/q_d(v_d)),
 *       v_d = argmax p_d (vso_reference_logkappa).
 *   Tree (App. E verification): node n's token was drafted from the row of
 *   parent(n); alpha_n uses that row; A_n = a_n AND A_parent(n); a rejected node
 *   whose parent is accepted gets a residual token drawn at the parent's row.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ */
/* Step O1: next-token distributions at temperature T (Eq. 1, Sec. 3). */
/* lp[v] = x_v/T - log sum_j exp(x_j/T), computed with the max shifted out. */
static double log_softmax_row(const float* x, int64_t V, double T, double* lp)
{
    double M = -INFINITY;
    for (int64_t v = 0; v < V; ++v) {
        double a = (double)x[v] / T;
        if (a > M) M = a;
    }
    double Z = 0.0;
    for (int64_t v = 0; v < V; ++v) Z += exp((double)x[v] / T - M);
    double lse = M + log(Z);
    for (int64_t v = 0; v < V; ++v) lp[v] = (double)x[v] / T - lse;
    return lse; /* log-partition of the row at temperature T */
}

/* Inverse-CDF draw: smallest v with u < F(v) = sum_{j<=v} prob[j].  If
 * rounding leaves no such v, the largest v with prob[v] > 0.  *margin is the
 * distance from u to the nearest boundary of the chosen interval. */
static int64_t sample_inverse_cdf(const double* prob, int64_t V, double u, double* margin)
{
    double F = 0.0;
    for (int64_t v = 0; v < V; ++v) {
        double Fprev = F;
        F += prob[v];
        if (u < F) {
            double m1 = u - Fprev, m2 = F - u;
            *margin = m1 < m2 ? m1 : m2;
            return v;
        }
    }
    for (int64_t v = V - 1; v >= 0; --v)
        if (prob[v] > 0.0) { *margin = 0.0; return v; }
    *margin = 0.0;
    return 0;
}

/* The T -> 0 limit of softmax(x / T) (R12): one-hot at the first maximum. */
static int64_t greedy_one_hot(const float* x, int64_t V, double* prob)
{
    int64_t m = 0;
    for (int64_t v = 1; v < V; ++v) if (x[v] > x[m]) m = v;
    for (int64_t v = 0; v < V; ++v) prob[v] = v == m ? 1.0 : 0.0;
    return m;
}

/* The distributions of one row that the decisions use: exp of the
 * log-probabilities at T > 0, the one-hot limits at T = 0 (R12). */
static void decision_dists(const float* xq, const float* xp, int64_t V, int greedy,
                           const double* lq, const double* lp, double* q, double* p)
{
    if (greedy) {
        greedy_one_hot(xq, V, q);
        greedy_one_hot(xp, V, p);
    } else {
        for (int64_t v = 0; v < V; ++v) { q[v] = exp(lq[v]); p[v] = exp(lp[v]); }
    }
}

/* ------------------------------------------------------------------ */
/* Inputs / outputs of the linear-path oracle.  Pointers may be NULL where
 * marked optional.  All per-row arrays have R = B*K*D entries. */
typedef struct {
    const float* draft;        /* [R][V] draft logits (exact input values)   */
    const float* target;       /* [R][V] target logits                       */
    int32_t B, K, D;
    int64_t V;
    double T;                  /* temperature, > 0                           */
    const float* u_draft;      /* [R] uniforms for z~ ~ q                    */
    const float* u_accept;     /* [R] uniforms r of Eq. 1                    */
    const float* u_correct;    /* [R] uniforms for the correction            */
    const float* ref_logkappa; /* optional [B][D]: log k(z-bar_{<=l})        */
    double w_base;             /* w(l) = w_base^l                            */
    double tau_car;            /* CAR temperature tau                        */
    int32_t zeta_mode;         /* 0: q(path) (literal), 1: log q(path)       */
    double kl_weight;          /* weight of the top-K term (R11), 0 = none   */
    int32_t kl_topk;           /* K of Eq. klv (the paper's 10)              */
} vso_linear_in;

typedef struct {
    int32_t* tokens;        /* [R] z~                                   */
    double*  logq_tok;      /* [R] log q_{s,d}(z~_d)                    */
    double*  alpha;         /* [R] alpha_d = min(1, p/q) at z~_d        */
    uint8_t* accept;        /* [R] u_accept <= alpha                    */
    int32_t* accept_len;    /* [B*K] A_s                                */
    int32_t* corr_tokens;   /* [R] z'_d                                 */
    double*  logq_corr;     /* [R] log q_{s,d}(z'_d)                    */
    double*  alpha_corr;    /* [R] min(1, p/q) at z'_d                  */
    double*  logkappa;      /* [R] log k(z~_{<=l}),  l = d+1            */
    double*  logkappa_corr; /* [R] log k(z'_{<=l})                      */
    double*  logkappa_ref;  /* [R] log k(z-bar_{<=l})                   */
    int32_t* ref_tokens;    /* [R] v-bar_d (argmax of the target row)   */
    double*  expected_len;  /* [B*K] sum_k S_k (Eq. 11)                 */
    double*  row_lse;       /* [R][2] log-partition of q row, p row     */
    double*  weights;       /* [B][D][K][4]: o~, o', beta, zeta         */
    double*  loss;          /* [B+1]: loss_b, then the mean over b      */
    double*  grad;          /* optional [R][V] d loss / d draft logits  */
    double*  margins;       /* optional [R][6] decision margins (below) */
    double*  kl_loss;       /* optional [R] L_topK of the row (Eq. klv) */
} vso_linear_out;
/* margins[r][0]: draft sample, |u - nearest CDF boundary| of q
 * margins[r][1]: accept, |u_accept - alpha|
 * margins[r][2]: correction sample of z'_d (residual or p), +inf if none
 * margins[r][3]: o~ at l=d+1: decision_margin(log k(z~), log k(z-bar))
 * margins[r][4]: o' at l=d+1 when o~=0: decision_margin(log k(z'), log k(z-bar)),
 *                else +inf
 * margins[r][5]: alpha of the correction token, |alpha' - 1| is not a
 *                decision; kept +inf (reserved) */

/* The M-step given the E-step's discrete results.  Everything it needs per
 * prefix is a [D][K] table; it is split out so that the gradient can be
 * checked by finite differences with the weights held fixed (Eq. advance
 * treats o~, o', beta, zeta and N_b as constants). */

/* Oracle of Algorithm 2: w(l) * I[log k(z_{<=l}) >= log k(z-bar_{<=l})]. */
static double oracle_utility(double logk, double logk_ref, int l, double w_base)
{
    return (logk >= logk_ref) ? pow(w_base, (double)l) : 0.0;
}

/* Eq. beta (leave-one-out): sum_{j!=s} o'_j o~_j / sum_{j!=s} o'_j; 0 if the
 * denominator is 0 (reading R6). */
static double arw_beta(const double* ot, const double* op, int K, int s)
{
    double num = 0.0, den = 0.0;
    for (int j = 0; j < K; ++j) {
        if (j == s) continue;
        num += op[j] * ot[j];
        den += op[j];
    }
    return den > 0.0 ? num / den : 0.0;
}

/* Eq. zeta: softmax over the K proposals of c_j / tau, c_j = q(z~^{(j)}_{<=l})
 * (mode 0) or log q(z~^{(j)}_{<=l}) (mode 1).  The max is shifted out. */
static void car_zeta(const double* logq_path, int K, double tau, int mode, double* zeta)
{
    double* c = (double*)malloc(sizeof(double) * (size_t)K);
    double M = -INFINITY;
    for (int j = 0; j < K; ++j) {
        c[j] = (mode == 0 ? exp(logq_path[j]) : logq_path[j]) / tau;
        if (c[j] > M) M = c[j];
    }
    double Z = 0.0;
    for (int j = 0; j < K; ++j) Z += exp(c[j] - M);
    for (int j = 0; j < K; ++j) zeta[j] = exp(c[j] - M) / Z;
    free(c);
}

/* ------------------------------------------------------------------ */
/* Public: weights of one prefix from its E-step tables.  Tables are [D][K]
 * (l-major).  Outputs o~, o', beta, zeta as [D][K][4] and returns N_b.   */
double vso_prefix_weights(int K, int D,
                          const double* logkappa,      /* [K][D] log k(z~_{<=l})  */
                          const double* logkappa_corr, /* [K][D] log k(z'_{<=l})  */
                          const double* logkappa_ref,  /* [K][D] log k(zbar_{<=l})*/
                          const double* logq_path_tok, /* [K][D] log q(z~_{<=l})  */
                          double w_base, double tau_car, int zeta_mode,
                          double* weights /* [D][K][4] */)
{
    double N = 0.0;
    double* ot = (double*)malloc(sizeof(double) * (size_t)K);
    double* op = (double*)malloc(sizeof(double) * (size_t)K);
    double* lqp = (double*)malloc(sizeof(double) * (size_t)K);
    double* zeta = (double*)malloc(sizeof(double) * (size_t)K);
    for (int d = 0; d < D; ++d) {
        int l = d + 1;
        for (int s = 0; s < K; ++s) {
            double lk = logkappa[s * D + d], lkr = logkappa_ref[s * D + d];
            /* Algorithm 1: o~ = o(z~); keep z~ if o(z~) > 0 else substitute z'. */
            double o_tilde = oracle_utility(lk, lkr, l, w_base);
            ot[s] = o_tilde > 0.0 ? 1.0 : 0.0; /* binary validity (R5) */
            if (o_tilde > 0.0)
                op[s] = o_tilde; /* z = z~, o' = o(z~) */
            else
                op[s] = oracle_utility(logkappa_corr[s * D + d], lkr, l, w_base);
            lqp[s] = logq_path_tok[s * D + d];
            N += op[s];
        }
        car_zeta(lqp, K, tau_car, zeta_mode, zeta);
        for (int s = 0; s < K; ++s) {
            double* w = weights + ((size_t)d * K + s) * 4;
            w[0] = ot[s];
            w[1] = op[s];
            w[2] = arw_beta(ot, op, K, s);
            w[3] = zeta[s];
        }
    }
    free(ot); free(op); free(lqp); free(zeta);
    return N;
}

/* Public: J_b and the gradient of loss = -(1/B) J_b / N_b for one prefix with
 * the weights held fixed.  rows of this prefix: draft [K][D][V].
 * tokens/corr: [K][D]; weights [D][K][4].  Returns J_b; grad (optional)
 * is [K][D][V] and receives d(-(1/B) J_b/N_b)/d draft.  (Eq. advance.) */
double vso_prefix_objective(const float* draft, int K, int D, int64_t V, double T,
                            const int32_t* tokens, const int32_t* corr_tokens,
                            const double* weights, double N, int B_total,
                            double* grad)
{
    double* lq = (double*)malloc(sizeof(double) * (size_t)V * (size_t)(K * D));
    for (int s = 0; s < K; ++s)
        for (int d = 0; d < D; ++d)
            log_softmax_row(draft + ((size_t)s * D + d) * V, V, T, lq + ((size_t)s * D + d) * V);
    double J = 0.0;
    if (grad) memset(grad, 0, sizeof(double) * (size_t)V * (size_t)(K * D));
    for (int d = 0; d < D; ++d) {       /* l = d+1 */
        for (int s = 0; s < K; ++s) {
            const double* w = weights + ((size_t)d * K + s) * 4;
            double ot = w[0], op = w[1], beta = w[2], zeta = w[3];
            if (op == 0.0) continue;
            /* z^{(s,l)} = z~ if o~ = 1 else z' (Algorithm 1). */
            const int32_t* z = ot > 0.0 ? tokens : corr_tokens;
            double logq_z = 0.0, logq_zt = 0.0;
            for (int i = 0; i <= d; ++i) {
                logq_z += lq[((size_t)s * D + i) * V + z[s * D + i]];
                logq_zt += lq[((size_t)s * D + i) * V + tokens[s * D + i]];
            }
            J += op * (logq_z - beta * zeta * logq_zt);
            if (!grad || N <= 0.0) continue;
            /* d log q_i(t) / d x_{i,v} = (1[v=t] - q_i(v)) / T ; the loss is
             * -(1/B) J / N, so each term enters with -(1/(B N)). */
            double c_pos = -op / ((double)B_total * N);
            double c_neg = op * beta * zeta / ((double)B_total * N);
            for (int i = 0; i <= d; ++i) {
                const double* lqi = lq + ((size_t)s * D + i) * V;
                double* g = grad + ((size_t)s * D + i) * V;
                int32_t tz = z[s * D + i], tt = tokens[s * D + i];
                for (int64_t v = 0; v < V; ++v) {
                    double qv = exp(lqi[v]);
                    double d_pos = ((v == tz ? 1.0 : 0.0) - qv) / T;
                    double d_neg = ((v == tt ? 1.0 : 0.0) - qv) / T;
                    g[v] += c_pos * d_pos + c_neg * d_neg;
                }
            }
        }
    }
    free(lq);
    return J;
}

/* Margin of the decision log k(a_{<=l}) >= log k(b_{<=l}) (Algorithm 2), for
 * counting near-boundary decisions in tests.  log k is a sum of clipped
 * log-ratios min(0, r_i).  Unequal sums: the gap.  Equal sums: the decision
 * is exact when, at every position where the two paths hold different
 * tokens, both log-ratios are clipped (r >= 0); its margin is then the
 * smallest such r; any other equality is a coincidence (margin 0).  With an
 * input reference (rb == NULL) the sum b is a constant. */
static double decision_margin(double a, double b, int n, const double* ra, const int32_t* ta,
                              const double* rb, const int32_t* tb)
{
    if (a != b) return fabs(a - b);
    double m = INFINITY;
    for (int i = 0; i < n; ++i) {
        if (rb && ta[i] == tb[i]) continue; /* identical terms cancel exactly */
        if (ra[i] < 0.0) return 0.0;
        if (ra[i] < m) m = ra[i];
        if (rb) {
            if (rb[i] < 0.0) return 0.0;
            if (rb[i] < m) m = rb[i];
        }
    }
    if (!rb && b != 0.0) return 0.0;
    return m;
}

/* ------------------------------------------------------------------ */
/* VSD (KL), Eq. klv: the top-K renormalised cross-entropy of one row.  Omega
 * = the Kt tokens of highest target probability (lowest index on ties);
 * p^(x) = p(x) / sum_{y in Omega} p(y), q^ likewise;
 * L = -sum_{x in Omega} p^(x) log q^(x) (a term with p^(x) = 0 is 0).
 * tok[k] receives Omega in order of selection, dl[k] = dL/dx_{tok[k]} =
 * (q^ - p^)/T: log q^(x) = x_x/T - log sum_{Omega} exp(x_y/T), so the full
 * vocabulary's partition cancels and every other logit has derivative 0. */
static double topk_ce_row(const float* xq, const float* xp, int64_t V, double T, int Kt,
                          int32_t* tok, double* dl)
{
    if (Kt > V) Kt = (int)V;
    for (int k = 0; k < Kt; ++k) {
        int64_t best = -1;
        for (int64_t v = 0; v < V; ++v) {
            int taken = 0;
            for (int j = 0; j < k; ++j) taken |= tok[j] == v;
            if (taken) continue;
            if (best < 0 || xp[v] > xp[best]) best = v; /* strict: lowest index wins ties */
        }
        tok[k] = (int32_t)best;
    }
    double mp = -INFINITY, mq = -INFINITY;
    for (int k = 0; k < Kt; ++k) {
        double a = (double)xp[tok[k]] / T, b = (double)xq[tok[k]] / T;
        if (a > mp) mp = a;
        if (b > mq) mq = b;
    }
    double Sp = 0.0, Sq = 0.0;
    for (int k = 0; k < Kt; ++k) {
        Sp += exp((double)xp[tok[k]] / T - mp);
        Sq += exp((double)xq[tok[k]] / T - mq);
    }
    double L = 0.0;
    for (int k = 0; k < Kt; ++k) {
        double ph = exp((double)xp[tok[k]] / T - mp) / Sp;
        double lqh = (double)xq[tok[k]] / T - mq - log(Sq);
        if (ph > 0.0) L -= ph * lqh;
        dl[k] = (exp(lqh) - ph) / T;
    }
    return L;
}

/* ------------------------------------------------------------------ */
/* Public: the whole E-step + M-step for linear paths.  Returns 0 on success,
 * nonzero on an invalid argument. */
int vso_linear(const vso_linear_in* in, vso_linear_out* out)
{
    const int B = in->B, K = in->K, D = in->D;
    const int64_t V = in->V;
    if (B < 1 || K < 1 || D < 1 || V < 1 || !(in->T >= 0.0) || in->T == INFINITY) return 1;
    /* R12: T = 0 decides greedily; log q is then taken at temperature 1 */
    const int greedy = in->T == 0.0;
    const double T = greedy ? 1.0 : in->T;
    double* lq = (double*)malloc(sizeof(double) * (size_t)V);
    double* lp = (double*)malloc(sizeof(double) * (size_t)V);
    double* q = (double*)malloc(sizeof(double) * (size_t)V);
    double* p = (double*)malloc(sizeof(double) * (size_t)V);
    double* res = (double*)malloc(sizeof(double) * (size_t)V);
    /* per-prefix tables, [K][D] */
    double* lk = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double* lkc = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double* lkr = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double* lqpath = (double*)malloc(sizeof(double) * (size_t)(K * D));
    /* unclipped log-ratios log(p/q) at z~, z', v-bar (for decision margins) */
    double* rt = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double* rc = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double* rr = (double*)malloc(sizeof(double) * (size_t)(K * D));
    double loss_sum = 0.0;

    for (int b = 0; b < B; ++b) {
        /* ---------------- E-step (Algorithm 1), per proposal s ---------------- */
        for (int s = 0; s < K; ++s) {
            const size_t r0 = ((size_t)b * K + s) * D;
            int A = 0, still = 1;
            /* Draft the path z~ ~ q token by token and verify each token with
             * Eq. 1: alpha = min(1, p/q) at z~, accepted iff r <= alpha. */
            for (int d = 0; d < D; ++d) {
                const size_t r = r0 + d;
                const float* xq = in->draft + r * V;
                const float* xp = in->target + r * V;
                double lse_q = log_softmax_row(xq, V, T, lq);
                double lse_p = log_softmax_row(xp, V, T, lp);
                out->row_lse[2 * r + 0] = lse_q;
                out->row_lse[2 * r + 1] = lse_p;
                decision_dists(xq, xp, V, greedy, lq, lp, q, p);
                double mg;
                int64_t zt = sample_inverse_cdf(q, V, (double)in->u_draft[r], &mg);
                double alpha = p[zt] / q[zt];
                if (alpha > 1.0) alpha = 1.0;
                double u = (double)in->u_accept[r];
                uint8_t a = (u <= alpha) ? 1 : 0;
                out->tokens[r] = (int32_t)zt;
                out->logq_tok[r] = lq[zt];
                out->alpha[r] = alpha;
                out->accept[r] = a;
                if (out->margins) {
                    out->margins[6 * r + 0] = mg;
                    out->margins[6 * r + 1] = fabs(u - alpha);
                    out->margins[6 * r + 2] = INFINITY;
                    out->margins[6 * r + 5] = INFINITY;
                }
                if (still && a) A = d + 1; else still = 0;
                /* Greedy reference token of Algorithm 2 (reading R4). */
                int64_t vb = 0;
                for (int64_t v = 1; v < V; ++v) if (xp[v] > xp[vb]) vb = v;
                double ab = p[vb] / q[vb];
                if (ab > 1.0) ab = 1.0;
                out->ref_tokens[r] = (int32_t)vb;
                rt[s * D + d] = log(p[zt] / q[zt]);
                rr[s * D + d] = log(p[vb] / q[vb]);
                /* prefix sums over l: log k(z~_{<=l}) = sum_{i<=l} log alpha_i (Eq. 2) */
                double prev = d ? lk[s * D + d - 1] : 0.0;
                lk[s * D + d] = prev + log(alpha);
                double prevr = d ? lkr[s * D + d - 1] : 0.0;
                lkr[s * D + d] = prevr + log(ab);
                double prevq = d ? lqpath[s * D + d - 1] : 0.0;
                lqpath[s * D + d] = prevq + lq[zt];
            }
            out->accept_len[(size_t)b * K + s] = A;
            /* Expected accepted length, Eq. 11: sum_{k=1..D} S_k. */
            double EA = 0.0;
            for (int d = 0; d < D; ++d) EA += exp(lk[s * D + d]);
            out->expected_len[(size_t)b * K + s] = EA;

            /* Correction (Sec. 3 + reading R3): z'_d = z~_d for d < A; at the
             * first rejection a residual token from norm(max(0, p - q)); after
             * it, p-samples from the given rows. */
            for (int d = 0; d < D; ++d) {
                const size_t r = r0 + d;
                int64_t zc;
                double mg = INFINITY;
                log_softmax_row(in->draft + r * V, V, T, lq);
                log_softmax_row(in->target + r * V, V, T, lp);
                decision_dists(in->draft + r * V, in->target + r * V, V, greedy, lq, lp, q, p);
                if (d < A) {
                    zc = out->tokens[r];
                } else if (d == A) {
                    double Rm = 0.0;
                    for (int64_t v = 0; v < V; ++v) {
                        double dv = p[v] - q[v];
                        res[v] = dv > 0.0 ? dv : 0.0;
                        Rm += res[v];
                    }
                    if (Rm > 0.0) {
                        for (int64_t v = 0; v < V; ++v) res[v] /= Rm;
                        zc = sample_inverse_cdf(res, V, (double)in->u_correct[r], &mg);
                    } else {
                        zc = sample_inverse_cdf(p, V, (double)in->u_correct[r], &mg); /* R10 */
                    }
                } else {
                    zc = sample_inverse_cdf(p, V, (double)in->u_correct[r], &mg);
                }
                double ac = p[zc] / q[zc];
                if (ac > 1.0) ac = 1.0;
                out->corr_tokens[r] = (int32_t)zc;
                out->logq_corr[r] = lq[zc];
                out->alpha_corr[r] = ac;
                rc[s * D + d] = log(p[zc] / q[zc]);
                if (out->margins) out->margins[6 * r + 2] = mg;
                double prev = d ? lkc[s * D + d - 1] : 0.0;
                lkc[s * D + d] = prev + log(ac);
            }
            if (in->ref_logkappa)
                for (int d = 0; d < D; ++d)
                    lkr[s * D + d] = (double)in->ref_logkappa[(size_t)b * D + d];
            for (int d = 0; d < D; ++d) {
                const size_t r = r0 + d;
                out->logkappa[r] = lk[s * D + d];
                out->logkappa_corr[r] = lkc[s * D + d];
                out->logkappa_ref[r] = lkr[s * D + d];
            }
        }

        /* ---------------- M-step: weights, loss, gradient ---------------- */
        double* wb = out->weights + (size_t)b * D * K * 4;
        double N = vso_prefix_weights(K, D, lk, lkc, lkr, lqpath, in->w_base, in->tau_car,
                                      in->zeta_mode, wb);
        if (out->margins) {
            const int32_t* tz = out->tokens + (size_t)b * K * D;
            const int32_t* tc = out->corr_tokens + (size_t)b * K * D;
            const int32_t* tr = out->ref_tokens + (size_t)b * K * D;
            const int refin = in->ref_logkappa != NULL;
            for (int s = 0; s < K; ++s)
                for (int d = 0; d < D; ++d) {
                    const size_t r = ((size_t)b * K + s) * D + d;
                    const int o = s * D;
                    out->margins[6 * r + 3] =
                        decision_margin(lk[o + d], lkr[o + d], d + 1, rt + o, tz + o,
                                        refin ? NULL : rr + o, tr + o);
                    out->margins[6 * r + 4] =
                        wb[((size_t)d * K + s) * 4 + 0] > 0.0
                            ? INFINITY
                            : decision_margin(lkc[o + d], lkr[o + d], d + 1, rc + o, tc + o,
                                              refin ? NULL : rr + o, tr + o);
                }
        }
        const size_t rb = (size_t)b * K * D;
        double J = vso_prefix_objective(in->draft + rb * V, K, D, V, T,
                                        out->tokens + rb, out->corr_tokens + rb, wb, N, B,
                                        out->grad ? out->grad + rb * V : NULL);
        double lb = N > 0.0 ? -J / N : 0.0;
        if (in->kl_weight != 0.0) {
            /* R11: + kl_weight (1/S) sum over the prefix's rows of Eq. klv */
            int32_t tok[64];
            double dl[64];
            int Kt = in->kl_topk < 1 ? 1 : (in->kl_topk > 64 ? 64 : in->kl_topk);
            double kl = 0.0;
            for (size_t r = rb; r < rb + (size_t)K * D; ++r) {
                double L = topk_ce_row(in->draft + r * V, in->target + r * V, V, T, Kt, tok, dl);
                if (out->kl_loss) out->kl_loss[r] = L;
                kl += L;
                if (out->grad) {
                    int kk = Kt > V ? (int)V : Kt;
                    for (int k = 0; k < kk; ++k)
                        out->grad[r * V + tok[k]] += in->kl_weight / ((double)B * K) * dl[k];
                }
            }
            lb += in->kl_weight * kl / (double)K;
        }
        out->loss[b] = lb;
        loss_sum += lb;
    }
    out->loss[B] = loss_sum / (double)B;
    free(lq); free(lp); free(q); free(p); free(res);
    free(lk); free(lkc); free(lkr); free(lqpath); free(rt); free(rc); free(rr);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Tree verification (App. E tree, Eq. 1 per node).  Rows are [B][N][V]:
 * row (b,n) holds the distributions that node n's children were drafted
 * from.  parent[b][0] = -1 (root, no token); parent[b][n] < n otherwise. */
typedef struct {
    const float* draft;
    const float* target;
    int32_t B, N;
    int64_t V;
    double T;
    const int32_t* parent;     /* [B][N] */
    const int32_t* tokens;     /* [B][N] token of node n (n >= 1)      */
    const float* u_accept;     /* [B][N] */
    const float* u_correct;    /* [B][N] */
    int32_t rule;              /* 0: independent per branch; 1: sequential siblings (R14) */
} vso_tree_in;

typedef struct {
    double*  alpha;        /* [B][N] min(1, p/q) at the parent's row; root 1 */
    uint8_t* accept;       /* [B][N] u_accept <= alpha; root 1              */
    uint8_t* path_accept;  /* [B][N] A_n = a_n AND A_parent                 */
    double*  logkappa;     /* [B][N] sum of log alpha along the path        */
    int32_t* corr_tokens;  /* [B][N] residual token at the parent's row for
                              a rejected node with an accepted parent, -1 else */
    int32_t* deepest;      /* [B] deepest accepted node (lowest index ties) */
    int32_t* accept_len;   /* [B] depth of the deepest accepted node        */
    int32_t* bonus;        /* [B] token emitted after the accepted path      */
    double*  margins;      /* optional [B][N][2]: accept, correction sample */
} vso_tree_out;

/* R14: the sequential sibling rule.  Scratch buffers of V (lq, lp, q, p,
 * res) and N (depth) are the caller's. */
static int tree_sequential(const vso_tree_in* in, vso_tree_out* out, double* lq, double* lp,
                           double* q, double* p, double* res, int* depth)
{
    const int B = in->B, N = in->N;
    const int64_t V = in->V;
    const double T = in->T;
    for (int b = 0; b < B; ++b) {
        const int32_t* par = in->parent + (size_t)b * N;
        const size_t n0 = (size_t)b * N;
        if (par[0] != -1) return 2;
        depth[0] = 0;
        for (int n = 1; n < N; ++n) {
            if (par[n] < 0 || par[n] >= n) return 2;
            depth[n] = depth[par[n]] + 1;
        }
        for (int n = 0; n < N; ++n) {
            out->alpha[n0 + n] = n ? 0.0 : 1.0;
            out->accept[n0 + n] = n ? 0 : 1;
            out->path_accept[n0 + n] = n ? 0 : 1;
            out->corr_tokens[n0 + n] = -1;
            if (out->margins) {
                out->margins[2 * (n0 + n)] = INFINITY;
                out->margins[2 * (n0 + n) + 1] = INFINITY;
            }
        }
        /* log kappa: the path validity of Eq. 2, independent ratios along the path */
        out->logkappa[n0] = 0.0;
        for (int n = 1; n < N; ++n) {
            const size_t rp = n0 + (size_t)par[n];
            log_softmax_row(in->draft + rp * V, V, T, lq);
            log_softmax_row(in->target + rp * V, V, T, lp);
            const int32_t t = in->tokens[n0 + n];
            double a = exp(lp[t]) / exp(lq[t]);
            if (a > 1.0) a = 1.0;
            out->logkappa[n0 + n] = out->logkappa[rp] + log(a);
        }
        /* the accepted path, node by node (parents come first) */
        for (int u = 0; u < N; ++u) {
            if (!out->path_accept[n0 + u]) continue;
            int last = -1;
            for (int n = u + 1; n < N; ++n) if (par[n] == u) last = n;
            if (last < 0) continue;
            const size_t ru = n0 + (size_t)u;
            log_softmax_row(in->draft + ru * V, V, T, lq);
            log_softmax_row(in->target + ru * V, V, T, lp);
            for (int64_t v = 0; v < V; ++v) { q[v] = exp(lq[v]); p[v] = exp(lp[v]); }
            for (int n = u + 1; n < N; ++n) {
                if (par[n] != u) continue;
                const int32_t t = in->tokens[n0 + n];
                double alpha;
                if (q[t] > 0.0) {
                    alpha = p[t] / q[t];
                    if (alpha > 1.0) alpha = 1.0;
                } else {
                    alpha = p[t] > 0.0 ? 1.0 : 0.0;
                }
                const double uu = (double)in->u_accept[n0 + n];
                const uint8_t a = (uu <= alpha) ? 1 : 0;
                out->alpha[n0 + n] = alpha;
                out->accept[n0 + n] = a;
                if (out->margins) out->margins[2 * (n0 + n)] = fabs(uu - alpha);
                if (a) {
                    out->path_accept[n0 + n] = 1;
                    break;
                }
                /* rejected: p <- norm(max(0, p - q)), q <- q without t */
                double Rm = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    const double dv = p[v] - q[v];
                    res[v] = dv > 0.0 ? dv : 0.0;
                    Rm += res[v];
                }
                if (Rm > 0.0)
                    for (int64_t v = 0; v < V; ++v) p[v] = res[v] / Rm;
                q[t] = 0.0;
                double Qs = 0.0;
                for (int64_t v = 0; v < V; ++v) Qs += q[v];
                for (int64_t v = 0; v < V; ++v) q[v] = Qs > 0.0 ? q[v] / Qs : 0.0;
                if (n == last) {  /* every child rejected: the correction token */
                    double mg;
                    out->corr_tokens[n0 + n] =
                        (int32_t)sample_inverse_cdf(p, V, (double)in->u_correct[n0 + n], &mg);
                    if (out->margins) out->margins[2 * (n0 + n) + 1] = mg;
                }
            }
        }
        /* the deepest accepted node; the bonus token after it */
        int best = 0;
        for (int n = 1; n < N; ++n)
            if (out->path_accept[n0 + n] && depth[n] > depth[best]) best = n;
        out->deepest[b] = best;
        out->accept_len[b] = depth[best];
        int last = -1;
        for (int n = best + 1; n < N; ++n) if (par[n] == best) last = n;
        int32_t bonus;
        if (last >= 0) {
            bonus = out->corr_tokens[n0 + last];
        } else {
            log_softmax_row(in->target + (n0 + best) * V, V, T, lp);
            for (int64_t v = 0; v < V; ++v) p[v] = exp(lp[v]);
            double mg;
            bonus = (int32_t)sample_inverse_cdf(p, V, (double)in->u_correct[n0 + best], &mg);
        }
        out->bonus[b] = bonus;
    }
    return 0;
}

int vso_tree(const vso_tree_in* in, vso_tree_out* out)
{
    const int B = in->B, N = in->N;
    const int64_t V = in->V;
    const double T = in->T;
    if (B < 1 || N < 1 || V < 1 || !(T > 0.0)) return 1;
    double* lq = (double*)malloc(sizeof(double) * (size_t)V);
    double* lp = (double*)malloc(sizeof(double) * (size_t)V);
    double* q = (double*)malloc(sizeof(double) * (size_t)V);
    double* p = (double*)malloc(sizeof(double) * (size_t)V);
    double* res = (double*)malloc(sizeof(double) * (size_t)V);
    int* depth = (int*)malloc(sizeof(int) * (size_t)N);
    int rc = 0;
    if (in->rule == 1) {
        rc = tree_sequential(in, out, lq, lp, q, p, res, depth);
        free(lq); free(lp); free(q); free(p); free(res); free(depth);
        return rc;
    }
    for (int b = 0; b < B && !rc; ++b) {
        const int32_t* par = in->parent + (size_t)b * N;
        const size_t n0 = (size_t)b * N;
        if (par[0] != -1) { rc = 2; break; }
        out->alpha[n0] = 1.0;
        out->accept[n0] = 1;
        out->path_accept[n0] = 1;
        out->logkappa[n0] = 0.0;
        out->corr_tokens[n0] = -1;
        depth[0] = 0;
        if (out->margins) { out->margins[2 * n0] = INFINITY; out->margins[2 * n0 + 1] = INFINITY; }
        for (int n = 1; n < N; ++n) {
            int pn = par[n];
            if (pn < 0 || pn >= n) { rc = 2; break; }
            depth[n] = depth[pn] + 1;
            const size_t rp = n0 + (size_t)pn; /* the parent's row */
            log_softmax_row(in->draft + rp * V, V, T, lq);
            log_softmax_row(in->target + rp * V, V, T, lp);
            for (int64_t v = 0; v < V; ++v) { q[v] = exp(lq[v]); p[v] = exp(lp[v]); }
            int32_t t = in->tokens[n0 + n];
            double alpha = p[t] / q[t];
            if (alpha > 1.0) alpha = 1.0;
            double u = (double)in->u_accept[n0 + n];
            uint8_t a = (u <= alpha) ? 1 : 0;
            out->alpha[n0 + n] = alpha;
            out->accept[n0 + n] = a;
            out->path_accept[n0 + n] = (uint8_t)(a && out->path_accept[rp]);
            out->logkappa[n0 + n] = out->logkappa[rp] + log(alpha);
            double mg = INFINITY;
            int32_t zc = -1;
            if (!a && out->path_accept[rp]) {
                double Rm = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    double dv = p[v] - q[v];
                    res[v] = dv > 0.0 ? dv : 0.0;
                    Rm += res[v];
                }
                if (Rm > 0.0) {
                    for (int64_t v = 0; v < V; ++v) res[v] /= Rm;
                    zc = (int32_t)sample_inverse_cdf(res, V, (double)in->u_correct[n0 + n], &mg);
                } else {
                    zc = (int32_t)sample_inverse_cdf(p, V, (double)in->u_correct[n0 + n], &mg);
                }
            }
            out->corr_tokens[n0 + n] = zc;
            if (out->margins) {
                out->margins[2 * (n0 + n)] = fabs(u - alpha);
                out->margins[2 * (n0 + n) + 1] = mg;
            }
        }
        if (rc) break;
        /* deepest accepted node, lowest index on ties */
        int best = 0;
        for (int n = 1; n < N; ++n)
            if (out->path_accept[n0 + n] && depth[n] > depth[best]) best = n;
        out->deepest[b] = best;
        out->accept_len[b] = depth[best];
        /* bonus token: the residual of the first rejected child of the
         * deepest node if it has children, otherwise a p-sample at its row. */
        int32_t bonus = -1;
        for (int n = 1; n < N; ++n)
            if (par[n] == best) { bonus = out->corr_tokens[n0 + n]; break; }
        if (bonus < 0) {
            log_softmax_row(in->target + (n0 + best) * V, V, T, lp);
            for (int64_t v = 0; v < V; ++v) p[v] = exp(lp[v]);
            double mg;
            bonus = (int32_t)sample_inverse_cdf(p, V, (double)in->u_correct[n0 + best], &mg);
        }
        out->bonus[b] = bonus;
    }
    free(lq); free(lp); free(q); free(p); free(res); free(depth);
    return rc;
}

/* ------------------------------------------------------------------ */
/* R15: the E-step + M-step over draft trees, every node a latent proposal.  */
typedef struct {
    const float* draft;
    const float* target;
    int32_t B, N;
    int64_t V;
    double T;
    const int32_t* parent;     /* [B][N] */
    const int32_t* tokens;     /* [B][N] */
    const float* u_accept;     /* [B][N] */
    const float* u_correct;    /* [B][N] */
    double w_base, tau_car;
    int32_t zeta_mode;
} vso_tree_em_in;

typedef struct {
    int32_t* corr_tokens;   /* [B][N] z'_x (root -1)                          */
    double* logq_tok;       /* [B][N] log q_{par(x)}(t_x) (root 0)            */
    double* logq_corr;      /* [B][N] log q_{par(x)}(z'_x)                     */
    double* logkappa;       /* [B][N] sum of log alpha on the root path        */
    double* logkappa_corr;  /* [B][N] of log alpha' (z')                       */
    double* logkappa_ref;   /* [B][N] of log alpha-bar (the rows' argmaxes)    */
    double* weights;        /* [B][N][4] o~, o', beta, zeta (root 0)           */
    double* loss;           /* [B+1]                                          */
    double* grad;           /* optional [B*N][V]                              */
    double* margins;        /* optional [B][N][3]: accept, z' draw, o~        */
} vso_tree_em_out;

int vso_tree_em(const vso_tree_em_in* in, vso_tree_em_out* out)
{
    const int B = in->B, N = in->N;
    const int64_t V = in->V;
    const double T = in->T;
    if (B < 1 || N < 1 || V < 1 || !(T > 0.0)) return 1;
    double* lq = (double*)malloc(sizeof(double) * (size_t)V);
    double* lp = (double*)malloc(sizeof(double) * (size_t)V);
    double* q = (double*)malloc(sizeof(double) * (size_t)V);
    double* p = (double*)malloc(sizeof(double) * (size_t)V);
    double* res = (double*)malloc(sizeof(double) * (size_t)V);
    double* lqall = (double*)malloc(sizeof(double) * (size_t)V * (size_t)N); /* log q per row */
    int* depth = (int*)malloc(sizeof(int) * (size_t)N);
    uint8_t* pacc = (uint8_t*)malloc((size_t)N);
    double* lqpath = (double*)malloc(sizeof(double) * (size_t)N);
    double* lcpath = (double*)malloc(sizeof(double) * (size_t)N);
    int* grp = (int*)malloc(sizeof(int) * (size_t)N);
    double* ot = (double*)malloc(sizeof(double) * (size_t)N);
    double* op = (double*)malloc(sizeof(double) * (size_t)N);
    double* lqz = (double*)malloc(sizeof(double) * (size_t)N);
    double* zeta = (double*)malloc(sizeof(double) * (size_t)N);
    double loss_sum = 0.0;
    int rc = 0;
    for (int b = 0; b < B && !rc; ++b) {
        const int32_t* par = in->parent + (size_t)b * N;
        const size_t n0 = (size_t)b * N;
        if (par[0] != -1) { rc = 2; break; }
        depth[0] = 0;
        for (int n = 1; n < N; ++n) {
            if (par[n] < 0 || par[n] >= n) { rc = 2; break; }
            depth[n] = depth[par[n]] + 1;
        }
        if (rc) break;
        for (int n = 0; n < N; ++n)
            log_softmax_row(in->draft + (n0 + n) * V, V, T, lqall + (size_t)n * V);
        double* W = out->weights + n0 * 4;
        for (int i = 0; i < 4 * N; ++i) W[i] = 0.0;
        /* E-step per position x (R15 with R3, R4): the token's test at its
         * parent's row, the corrected token, the reference of that row */
        pacc[0] = 1;
        out->corr_tokens[n0] = -1;
        out->logq_tok[n0] = out->logq_corr[n0] = 0.0;
        out->logkappa[n0] = out->logkappa_corr[n0] = out->logkappa_ref[n0] = 0.0;
        lqpath[0] = lcpath[0] = 0.0;
        if (out->margins)
            for (int k = 0; k < 3; ++k) out->margins[3 * n0 + k] = INFINITY;
        for (int x = 1; x < N; ++x) {
            const int a = par[x];
            const size_t ra = n0 + (size_t)a;
            const double* lqa = lqall + (size_t)a * V;
            log_softmax_row(in->target + ra * V, V, T, lp);
            for (int64_t v = 0; v < V; ++v) { q[v] = exp(lqa[v]); p[v] = exp(lp[v]); }
            const int32_t t = in->tokens[n0 + x];
            double alpha = p[t] / q[t];
            if (alpha > 1.0) alpha = 1.0;
            const double u = (double)in->u_accept[n0 + x];
            const int acc = u <= alpha;
            pacc[x] = (uint8_t)(acc && pacc[a]);
            double mg = INFINITY;
            int64_t zc;
            if (pacc[x]) {
                zc = t;
            } else if (pacc[a]) { /* the first rejection on the path: residual */
                double Rm = 0.0;
                for (int64_t v = 0; v < V; ++v) {
                    const double dv = p[v] - q[v];
                    res[v] = dv > 0.0 ? dv : 0.0;
                    Rm += res[v];
                }
                if (Rm > 0.0) {
                    for (int64_t v = 0; v < V; ++v) res[v] /= Rm;
                    zc = sample_inverse_cdf(res, V, (double)in->u_correct[n0 + x], &mg);
                } else {
                    zc = sample_inverse_cdf(p, V, (double)in->u_correct[n0 + x], &mg);
                }
            } else { /* below a rejection: a draw from p */
                zc = sample_inverse_cdf(p, V, (double)in->u_correct[n0 + x], &mg);
            }
            double ac = p[zc] / q[zc];
            if (ac > 1.0) ac = 1.0;
            int64_t vb = 0;
            const float* xp = in->target + ra * V;
            for (int64_t v = 1; v < V; ++v) if (xp[v] > xp[vb]) vb = v;
            double ab = p[vb] / q[vb];
            if (ab > 1.0) ab = 1.0;
            out->corr_tokens[n0 + x] = (int32_t)zc;
            out->logq_tok[n0 + x] = lqa[t];
            out->logq_corr[n0 + x] = lqa[zc];
            out->logkappa[n0 + x] = out->logkappa[ra] + log(alpha);
            out->logkappa_corr[n0 + x] = out->logkappa_corr[ra] + log(ac);
            out->logkappa_ref[n0 + x] = out->logkappa_ref[ra] + log(ab);
            lqpath[x] = lqpath[a] + lqa[t];
            lcpath[x] = lcpath[a] + lqa[zc];
            if (out->margins) {
                out->margins[3 * (n0 + x)] = fabs(u - alpha);
                out->margins[3 * (n0 + x) + 1] = mg;
            }
        }
        /* M-step: o~, o' per proposal (Algorithm 2 with w(depth)) */
        double Nb = 0.0;
        for (int n = 1; n < N; ++n) {
            const double lk = out->logkappa[n0 + n], lkr = out->logkappa_ref[n0 + n];
            const double o_tilde = oracle_utility(lk, lkr, depth[n], in->w_base);
            W[4 * n + 0] = o_tilde > 0.0 ? 1.0 : 0.0;
            W[4 * n + 1] = o_tilde > 0.0 ? o_tilde
                                          : oracle_utility(out->logkappa_corr[n0 + n], lkr,
                                                           depth[n], in->w_base);
            Nb += W[4 * n + 1];
            if (out->margins) {
                const double d = lk - lkr;
                out->margins[3 * (n0 + n) + 2] = d == 0.0 ? 0.0 : fabs(d);
            }
        }
        /* beta, zeta over the proposals of one length (the nodes of one depth) */
        int maxd = 0;
        for (int n = 1; n < N; ++n) if (depth[n] > maxd) maxd = depth[n];
        for (int l = 1; l <= maxd; ++l) {
            int m = 0;
            for (int n = 1; n < N; ++n)
                if (depth[n] == l) {
                    grp[m] = n;
                    ot[m] = W[4 * n + 0];
                    op[m] = W[4 * n + 1];
                    lqz[m] = lqpath[n];
                    ++m;
                }
            if (m == 0) continue;
            car_zeta(lqz, m, in->tau_car, in->zeta_mode, zeta);
            for (int i = 0; i < m; ++i) {
                W[4 * grp[i] + 2] = arw_beta(ot, op, m, i);
                W[4 * grp[i] + 3] = zeta[i];
            }
        }
        /* the objective (Eq. advance) and its gradient */
        double J = 0.0;
        double* G = out->grad ? out->grad + n0 * V : NULL;
        if (G) memset(G, 0, sizeof(double) * (size_t)N * (size_t)V);
        for (int n = 1; n < N; ++n) {
            const double o_t = W[4 * n], o_p = W[4 * n + 1], beta = W[4 * n + 2], z = W[4 * n + 3];
            if (o_p == 0.0) continue;
            const double lqn = o_t > 0.0 ? lqpath[n] : lcpath[n];
            J += o_p * (lqn - beta * z * lqpath[n]);
            if (!G || Nb <= 0.0) continue;
            const double c_pos = -o_p / ((double)B * Nb);
            const double c_neg = o_p * beta * z / ((double)B * Nb);
            for (int x = n; x > 0; x = par[x]) { /* the positions of the path */
                const int a = par[x];
                const double* lqa = lqall + (size_t)a * V;
                double* g = G + (size_t)a * V;
                const int32_t tz = o_t > 0.0 ? in->tokens[n0 + x] : out->corr_tokens[n0 + x];
                const int32_t tt = in->tokens[n0 + x];
                for (int64_t v = 0; v < V; ++v) {
                    const double qv = exp(lqa[v]);
                    g[v] += c_pos * ((v == tz ? 1.0 : 0.0) - qv) / T +
                            c_neg * ((v == tt ? 1.0 : 0.0) - qv) / T;
                }
            }
        }
        const double lb = Nb > 0.0 ? -J / Nb : 0.0;
        out->loss[b] = lb;
        loss_sum += lb;
    }
    if (!rc) out->loss[B] = loss_sum / (double)B;
    free(lq); free(lp); free(q); free(p); free(res); free(lqall); free(depth); free(pacc);
    free(lqpath); free(lcpath); free(grp); free(ot); free(op); free(lqz); free(zeta);
    return rc;
}

/* ------------------------------------------------------------------ */
/* R13: log kappa of a supplied greedy reference path (Algorithm 2).  Rows
 * [B][D][V] of the draft and target along z-bar; out [B][D] receives
 * sum_{d<=l} log min(1, p_d(v_d) / q_d(v_d)), v_d = argmax p_d (lowest index
 * on ties), at temperature T (T = 0: the one-hot limits, R12). */
int vso_reference_logkappa(const float* draft, const float* target, int32_t B, int32_t D,
                           int64_t V, double T, double* out)
{
    if (B < 1 || D < 1 || V < 1 || !(T >= 0.0) || T == INFINITY) return 1;
    const int greedy = T == 0.0;
    double* lq = (double*)malloc(sizeof(double) * (size_t)V);
    double* lp = (double*)malloc(sizeof(double) * (size_t)V);
    double* q = (double*)malloc(sizeof(double) * (size_t)V);
    double* p = (double*)malloc(sizeof(double) * (size_t)V);
    for (int b = 0; b < B; ++b) {
        double acc = 0.0;
        for (int d = 0; d < D; ++d) {
            const size_t r = (size_t)b * D + d;
            const float* xq = draft + r * V;
            const float* xp = target + r * V;
            log_softmax_row(xq, V, greedy ? 1.0 : T, lq);
            log_softmax_row(xp, V, greedy ? 1.0 : T, lp);
            decision_dists(xq, xp, V, greedy, lq, lp, q, p);
            int64_t vb = 0;
            for (int64_t v = 1; v < V; ++v) if (xp[v] > xp[vb]) vb = v;
            double ab = p[vb] / q[vb];
            if (ab > 1.0) ab = 1.0;
            acc += log(ab);
            out[r] = acc;
        }
    }
    free(lq); free(lp); free(q); free(p);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Small public pieces used by the pins. */
double vso_log_softmax(const float* x, int64_t V, double T, double* lp)
{
    return log_softmax_row(x, V, T, lp);
}

int64_t vso_sample(const double* prob, int64_t V, double u, double* margin)
{
    return sample_inverse_cdf(prob, V, u, margin);
}

/* Eq. klv for one row (see topk_ce_row). */
double vso_topk_ce(const float* xq, const float* xp, int64_t V, double T, int Kt, int32_t* tok,
                   double* dl)
{
    return topk_ce_row(xq, xp, V, T, Kt, tok, dl);
}

/* The margin of one Algorithm 2 comparison (see decision_margin); rb and tb
 * may be NULL (an input reference). */
double vso_decision_margin(double a, double b, int n, const double* ra, const int32_t* ta,
                           const double* rb, const int32_t* tb)
{
    return decision_margin(a, b, n, ra, ta, rb, tb);
}
