/*
 * osd_oracle.c -- plain, slow, double-precision CPU oracle for the two per-step
 * operations of Online Speculative Decoding (Liu et al., "Online Speculative
 * Decoding", ICML 2024):
 *
 *   osd_oracle_verify   speculative-sampling verification (Appendix A.1,
 *                       the accept rule and the residual distribution p'(y);
 *                       Algorithm 1, "Determine number of accepted tokens")
 *   osd_oracle_distill  per-position distance D(p || q_theta) of Eq. 2 / Eq. 3
 *                       (forward KL, reverse KL, JSD[beta]) plus total
 *                       variation distance, and the analytic gradient with
 *                       respect to the draft logits (Algorithm 1, "Update
 *                       q_theta ... analytically").
 *   osd_oracle_verify_tree  multi-candidate verification over a token tree
 *                       (the tree-style decoding of the paper's Medusa study).
 *   osd_oracle_mixed_sample  one draw per position from the mixture
 *                       beta p + (1 - beta) q_theta (Section 4.1, mixed
 *                       sampling of the tokens the distillation is run on).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline leg of bench.py may load this library.  It shares no code,
 * header, table or constant with the CUDA library and never calls it.
 *
 * Everything is computed in double precision, one row at a time, with
 * sequential sums in ascending vocabulary order.  Inputs arrive as double
 * arrays; bf16 and fp32 logits convert to double exactly.
 *
 * Readings of the paper that the code fixes (the paper is silent on them):
 *   - accept test is strict: accept y_i iff u_i < r_i, r_i = p_i(y_i)/q_i(y_i)
 *     computed as exp(log p - log q); identical to u < min(1, r) for u < 1.
 *   - q(y_i) = 0 with p(y_i) > 0 gives r = +inf (accept); both zero gives
 *     r = 0 (reject).
 *   - uniforms[b, 0..k-1] are the k accept tests, uniforms[b, k] is the one
 *     inverse-CDF draw for the residual (a < k) or bonus (a = k) sample.
 *   - inverse CDF: ascending index, j* = min{ j : C_j > u*W }; if rounding
 *     leaves no such j, the largest j with w_j > 0; if W = 0, argmax of p
 *     (lowest index).
 *   - temperature scales both draft and target logits; T = 0 is greedy
 *     (argmax-prefix matching, lowest index on ties, uniforms ignored).
 *   - any draft token outside [0, V) marks the whole sequence bad:
 *     accepted = -1, out_tokens = -1, mask = 0, diagnostics NaN.
 *   - the mismatch mask marks only the first rejected position (a < k).
 *   - distill applies one temperature tau to both rows (Section 4.1: the
 *     logits are divided by tau before the softmax) and returns the
 *     per-position loss and its gradient with respect to the raw draft
 *     logits (hence a factor 1/tau); inactive rows get loss 0 and their
 *     gradient row is left untouched.
 *   - the label fine-tuning loss (FT of Table 1) is the cross-entropy of q
 *     to the target's argmax label, lowest index on ties.
 *   - TVD = 1/2 sum |p - q|, subgradient with sign(0) = 0.
 *   - 0 * log 0 = 0: terms with zero probability contribute nothing.
 *
 * Parity pins for every function here live in tests/test_oracle_*.py
 * (closed forms, library routines, invariants, finite differences,
 * chi-square tests of the output distribution).
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>

/* Loss kinds; values are part of the oracle's own interface. */
enum { ORACLE_FKL = 0, ORACLE_RKL = 1, ORACLE_JSD = 2, ORACLE_TVD = 3, ORACLE_CE = 4 };

/* log-softmax of x[0..V-1] / T into out (T > 0). Eq. 3 / Section 4.1
 * "softmax with temperature": lp_j = x_j/T - log sum_i exp(x_i/T).      */
static void log_softmax(const double *x, long V, double T, double *out)
{
    double m = -INFINITY;
    for (long j = 0; j < V; ++j) {
        double s = x[j] / T;
        out[j] = s;
        if (s > m) m = s;
    }
    if (m == -INFINITY) {            /* every logit is -inf: no mass anywhere */
        for (long j = 0; j < V; ++j) out[j] = -INFINITY;
        return;
    }
    double sum = 0.0;
    for (long j = 0; j < V; ++j) sum += exp(out[j] - m);
    double lse = m + log(sum);
    for (long j = 0; j < V; ++j) out[j] = out[j] - lse;
}

/* Index of the largest element, lowest index on ties. */
static long argmax_first(const double *x, long V)
{
    long best = 0;
    for (long j = 1; j < V; ++j)
        if (x[j] > x[best]) best = j;
    return best;
}

/* Exported so tests can build expected distributions from the same oracle. */
void osd_oracle_log_softmax(const double *x, long V, double T, double *out)
{
    log_softmax(x, V, T, out);
}

/*
 * Speculative-sampling verification, Appendix A.1 and Algorithm 1.
 *
 * draft  [B, k, V]    draft logits  z (row i is q_theta(. | x, y_<i))
 * target [B, k+1, V]  target logits t (row i is p(. | x, y_<i))
 * tokens [B, k]       draft proposals y_1..y_k
 * uniforms [B, k+1]   u_1..u_k for the accept tests, u_{k+1} for the sample
 * T                   temperature (T = 0: greedy)
 * accepted [B], out_tokens [B, k+1], mask [B, k]
 * margin [B, k]       |u_i - r_i| for the positions decided; NaN after
 * cdf_gap [B]         min distance of u*W to the CDF step edges, / W
 * ratio [B, k]        r_i for the positions decided; NaN after (nullable)
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int osd_oracle_verify(const double *draft, const double *target,
                      long B, long k, long V,
                      const int32_t *tokens, const double *uniforms, double T,
                      int32_t *accepted, int32_t *out_tokens, uint8_t *mask,
                      double *margin, double *cdf_gap, double *ratio)
{
    if (B < 0 || k < 1 || V < 1 || !(T >= 0.0)) return -1;
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    double *lp = (double *)malloc(sizeof(double) * (size_t)V);
    double *w  = (double *)malloc(sizeof(double) * (size_t)V);
    if (!lq || !lp || !w) { free(lq); free(lp); free(w); return -1; }

    for (long b = 0; b < B; ++b) {
        const int32_t *y = tokens + b * k;
        const double *u = uniforms + b * (k + 1);
        int32_t *out = out_tokens + b * (k + 1);
        for (long i = 0; i < k; ++i) {
            mask[b * k + i] = 0;
            margin[b * k + i] = NAN;
            if (ratio) ratio[b * k + i] = NAN;
        }
        for (long i = 0; i <= k; ++i) out[i] = -1;
        cdf_gap[b] = NAN;

        int bad = 0;
        for (long i = 0; i < k; ++i)
            if (y[i] < 0 || y[i] >= V) bad = 1;
        if (bad) { accepted[b] = -1; continue; }

        long a = 0;
        long sample;
        if (T == 0.0) {
            /* Greedy: accept while the proposal is the target argmax. */
            while (a < k && y[a] == argmax_first(target + (b * (k + 1) + a) * V, V))
                ++a;
            sample = argmax_first(target + (b * (k + 1) + a) * V, V);
        } else {
            /* Accept test for i = 1..k in order, stop at the first reject. */
            while (a < k) {
                log_softmax(draft + (b * k + a) * V, V, T, lq);
                log_softmax(target + (b * (k + 1) + a) * V, V, T, lp);
                double lpy = lp[y[a]], lqy = lq[y[a]];
                double r;
                if (lqy == -INFINITY) r = (lpy > -INFINITY) ? INFINITY : 0.0;
                else r = exp(lpy - lqy);
                margin[b * k + a] = fabs(u[a] - r);
                if (ratio) ratio[b * k + a] = r;
                if (u[a] < r) ++a;
                else break;
            }
            /* The distribution of the extra token: p'(y) of Appendix A.1. */
            log_softmax(target + (b * (k + 1) + a) * V, V, T, lp);
            if (a < k) {
                log_softmax(draft + (b * k + a) * V, V, T, lq);
                for (long j = 0; j < V; ++j) {
                    double d = exp(lp[j]) - exp(lq[j]);
                    w[j] = d > 0.0 ? d : 0.0;       /* max(0, p - q) */
                }
            } else {
                for (long j = 0; j < V; ++j) w[j] = exp(lp[j]);
            }
            double W = 0.0;
            for (long j = 0; j < V; ++j) W += w[j];
            if (W > 0.0) {
                double tau = u[k] * W;               /* inverse CDF of w / W */
                double C = 0.0, Cprev = 0.0;
                sample = -1;
                for (long j = 0; j < V; ++j) {
                    Cprev = C;
                    C += w[j];
                    if (C > tau) { sample = j; break; }
                }
                if (sample < 0) {                    /* rounding left none */
                    for (long j = V - 1; j >= 0; --j)
                        if (w[j] > 0.0) { sample = j; break; }
                    Cprev = W - w[sample];
                    C = W;
                }
                double g1 = C - tau, g0 = tau - Cprev;
                cdf_gap[b] = (g1 < g0 ? g1 : g0) / W;
            } else {
                sample = argmax_first(lp, V);
            }
        }
        accepted[b] = (int32_t)a;
        for (long i = 0; i < a; ++i) out[i] = y[i];
        out[a] = (int32_t)sample;
        if (a < k) mask[b * k + a] = 1;
    }
    free(lq); free(lp); free(w);
    return 0;
}

/*
 * Per-position distillation loss and gradient, Eq. 2-3 (Section 4.1), with
 * softmax temperature tau, for every row n with mask[n] != 0 (mask may be NULL).
 *
 * draft, target [N, V]   logits z, t;  q = softmax(z/tau), p = softmax(t/tau)
 * kind                   0 FKL = KL(p||q), 1 RKL = KL(q||p),
 *                        2 JSD[beta] = beta KL(p||m) + (1-beta) KL(q||m),
 *                          m = beta p + (1-beta) q,
 *                        3 TVD = 1/2 sum |p - q|,
 *                        4 CE = -log q(y*), y* = argmax t (label fine-tuning)
 * loss [N]               per-position loss; 0 for inactive rows
 * dlogits [N, V]         d loss / d z (raw logits); inactive rows are not written
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int osd_oracle_distill(const double *draft, const double *target, long N, long V,
                       const uint8_t *mask, int kind, double beta, double tau,
                       double *loss, double *dlogits)
{
    if (N < 0 || V < 1 || kind < 0 || kind > 4) return -1;
    if (kind == ORACLE_JSD && !(beta >= 0.0 && beta <= 1.0)) return -1;
    if (!(tau > 0.0) || !isfinite(tau)) return -1;
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    double *lp = (double *)malloc(sizeof(double) * (size_t)V);
    if (!lq || !lp) { free(lq); free(lp); return -1; }

    for (long n = 0; n < N; ++n) {
        if (mask && !mask[n]) { loss[n] = 0.0; continue; }
        log_softmax(draft + n * V, V, tau, lq);
        log_softmax(target + n * V, V, tau, lp);
        double *g = dlogits + n * V;
        double l = 0.0;
        if (kind == ORACLE_FKL) {
            for (long j = 0; j < V; ++j) {
                double p = exp(lp[j]);
                if (p > 0.0) l += p * (lp[j] - lq[j]);
            }
            for (long j = 0; j < V; ++j) g[j] = exp(lq[j]) - exp(lp[j]);
        } else if (kind == ORACLE_RKL) {
            for (long j = 0; j < V; ++j) {
                double q = exp(lq[j]);
                if (q > 0.0) l += q * (lq[j] - lp[j]);
            }
            for (long j = 0; j < V; ++j) {
                double q = exp(lq[j]);
                g[j] = q > 0.0 ? q * ((lq[j] - lp[j]) - l) : 0.0;
            }
        } else if (kind == ORACLE_JSD) {
            double klp = 0.0, klq = 0.0;
            for (long j = 0; j < V; ++j) {
                double p = exp(lp[j]), q = exp(lq[j]);
                double m = beta * p + (1.0 - beta) * q;
                if (p > 0.0) klp += p * log(p / m);
                if (q > 0.0) klq += q * log(q / m);
            }
            if (beta > 0.0) l += beta * klp;
            if (beta < 1.0) l += (1.0 - beta) * klq;
            for (long j = 0; j < V; ++j) {
                double p = exp(lp[j]), q = exp(lq[j]);
                double m = beta * p + (1.0 - beta) * q;
                g[j] = (q > 0.0 && beta < 1.0)
                           ? (1.0 - beta) * q * (log(q / m) - klq) : 0.0;
            }
        } else if (kind == ORACLE_CE) {
            long ystar = argmax_first(target + n * V, V);
            l = -lq[ystar];
            for (long j = 0; j < V; ++j) g[j] = exp(lq[j]) - (j == ystar ? 1.0 : 0.0);
        } else { /* ORACLE_TVD */
            double G = 0.0;
            for (long j = 0; j < V; ++j) {
                double p = exp(lp[j]), q = exp(lq[j]);
                double s = (q > p) ? 0.5 : (q < p ? -0.5 : 0.0);
                l += 0.5 * fabs(p - q);
                G += q * s;
            }
            for (long j = 0; j < V; ++j) {
                double p = exp(lp[j]), q = exp(lq[j]);
                double s = (q > p) ? 0.5 : (q < p ? -0.5 : 0.0);
                g[j] = q * (s - G);
            }
        }
        /* the softmax sees z / tau, so d/dz carries a factor 1 / tau */
        for (long j = 0; j < V; ++j) g[j] /= tau;
        loss[n] = l;
    }
    free(lq); free(lp);
    return 0;
}

/*
 * Mixed-token sampling, Section 4.1: y ~ beta p + (1 - beta) q, with
 * p = softmax(t / tau) and q = softmax(z / tau) of one position, for each of
 * N rows (row n of the draft starts at draft + n*d_stride, of the target at
 * target + n*t_stride).  The draw is one inverse-CDF step over the mixture
 * weights w_j = beta p_j + (1 - beta) q_j in ascending vocabulary order, with
 * the conventions of the verify oracle's extra token: j* = min{ j : C_j > u W },
 * W = sum_j w_j; if rounding leaves no such j, the largest j with w_j > 0.
 *
 * uniforms [N]  u in [0, 1);  tokens [N] out;  cdf_gap [N] out (nullable):
 * distance of u W to the nearest edge of the chosen CDF step, divided by W.
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int osd_oracle_mixed_sample(const double *draft, const double *target, long N, long V,
                            long d_stride, long t_stride, const double *uniforms,
                            double beta, double tau, int32_t *tokens, double *cdf_gap)
{
    if (N < 0 || V < 1 || !(tau > 0.0) || !(beta >= 0.0 && beta <= 1.0)) return -1;
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    double *lp = (double *)malloc(sizeof(double) * (size_t)V);
    double *w  = (double *)malloc(sizeof(double) * (size_t)V);
    if (!lq || !lp || !w) { free(lq); free(lp); free(w); return -1; }
    for (long n = 0; n < N; ++n) {
        log_softmax(draft + n * d_stride, V, tau, lq);
        log_softmax(target + n * t_stride, V, tau, lp);
        double W = 0.0;
        for (long j = 0; j < V; ++j) {
            w[j] = beta * exp(lp[j]) + (1.0 - beta) * exp(lq[j]);
            W += w[j];
        }
        const double target_mass = uniforms[n] * W;
        double C = 0.0, Cprev = 0.0;
        long pick = -1;
        for (long j = 0; j < V; ++j) {
            Cprev = C;
            C += w[j];
            if (C > target_mass) { pick = j; break; }
        }
        if (pick < 0) {                              /* rounding left none */
            for (long j = V - 1; j >= 0; --j)
                if (w[j] > 0.0) { pick = j; break; }
            Cprev = W - w[pick];
            C = W;
        }
        tokens[n] = (int32_t)pick;
        if (cdf_gap) {
            double g1 = C - target_mass, g0 = target_mass - Cprev;
            cdf_gap[n] = (g1 < g0 ? g1 : g0) / W;
        }
    }
    free(lq); free(lp); free(w);
    return 0;
}

/*
 * Multi-candidate verification over a token tree: the tree-style speculative
 * decoding the paper runs OSD on with Medusa, where several candidates are
 * proposed per position.  Each node carries one candidate token; the children
 * of a node are the alternatives for the next position, tried in increasing
 * index order with the accept rule of Appendix A.1 applied to the current
 * residual: child y is accepted iff u < r(y) / q(y), starting from r = p; a
 * rejection replaces r by norm(max(0, r - q)) (multi-candidate speculative
 * sampling, which keeps the output distributed as p).  Accepting a child moves
 * the walk to it; when every child of the current node is rejected, or it has
 * none, one more token is drawn from r by the inverse CDF of the verify
 * oracle's extra token.  T = 0 is greedy: the first child equal to argmax p is
 * taken, and the extra token is argmax p.
 *
 * parent [n_nodes]         parent[0] = -1, 0 <= parent[i] < i (static tree)
 * draft  [B, n_nodes, V]   z at node i: the draft distribution q of node i's children
 * target [B, n_nodes, V]   t at node i: the target distribution p after node i's path
 * tokens [B, n_nodes]      candidate token of node i (node 0, the root, has none)
 * uniforms [B, n_nodes]    u[b, i] tests node i; u[b, 0] drives the extra draw
 * accepted [B]             accepted tokens (the depth reached); -1 if a token is
 *                          outside [0, V)
 * path [B, n_nodes]        the accepted nodes, root excluded, then -1
 * out_tokens [B, n_nodes]  the accepted tokens, the extra token, then -1
 * last_node [B]            the node where the walk stopped (-1 if bad)
 * margin [B, n_nodes]      |u - r(y)/q(y)| of every test made; NaN elsewhere
 * cdf_gap [B]              as in osd_oracle_verify; NaN at T = 0
 * Returns 0, or -1 on bad arguments / allocation failure.
 */
int osd_oracle_verify_tree(const double *draft, const double *target, long B, long n_nodes, long V,
                           const int32_t *parent, const int32_t *tokens, const double *uniforms,
                           double T, int32_t *accepted, int32_t *path, int32_t *out_tokens,
                           int32_t *last_node, double *margin, double *cdf_gap)
{
    if (B < 0 || n_nodes < 1 || V < 1 || !(T >= 0.0) || parent[0] != -1) return -1;
    for (long i = 1; i < n_nodes; ++i)
        if (parent[i] < 0 || parent[i] >= i) return -1;
    double *lq = (double *)malloc(sizeof(double) * (size_t)V);
    double *lp = (double *)malloc(sizeof(double) * (size_t)V);
    double *q = (double *)malloc(sizeof(double) * (size_t)V);
    double *r = (double *)malloc(sizeof(double) * (size_t)V);
    if (!lq || !lp || !q || !r) { free(lq); free(lp); free(q); free(r); return -1; }

    for (long b = 0; b < B; ++b) {
        const int32_t *y = tokens + b * n_nodes;
        const double *u = uniforms + b * n_nodes;
        int32_t *pth = path + b * n_nodes;
        int32_t *out = out_tokens + b * n_nodes;
        for (long i = 0; i < n_nodes; ++i) {
            pth[i] = -1;
            out[i] = -1;
            margin[b * n_nodes + i] = NAN;
        }
        cdf_gap[b] = NAN;
        int bad = 0;
        for (long i = 1; i < n_nodes; ++i)
            if (y[i] < 0 || y[i] >= V) bad = 1;
        if (bad) { accepted[b] = -1; last_node[b] = -1; continue; }

        long node = 0, depth = 0, extra = -1;
        for (;;) {
            const double *trow = target + (b * n_nodes + node) * V;
            long next = -1;
            if (T == 0.0) {
                long best = argmax_first(trow, V);
                for (long c = node + 1; c < n_nodes && next < 0; ++c)
                    if (parent[c] == node && y[c] == best) next = c;
                if (next < 0) { extra = best; break; }
            } else {
                log_softmax(trow, V, T, lp);
                log_softmax(draft + (b * n_nodes + node) * V, V, T, lq);
                for (long j = 0; j < V; ++j) { r[j] = exp(lp[j]); q[j] = exp(lq[j]); }
                for (long c = node + 1; c < n_nodes && next < 0; ++c) {
                    if (parent[c] != node) continue;
                    const double ry = r[y[c]], qy = q[y[c]];
                    double ratio;
                    if (qy > 0.0) ratio = ry / qy;
                    else ratio = (ry > 0.0) ? INFINITY : 0.0;
                    margin[b * n_nodes + c] = fabs(u[c] - ratio);
                    if (u[c] < ratio) {
                        next = c;
                    } else {                          /* r <- norm(max(0, r - q)) */
                        double W = 0.0;
                        for (long j = 0; j < V; ++j) {
                            const double d = r[j] - q[j];
                            r[j] = d > 0.0 ? d : 0.0;
                            W += r[j];
                        }
                        if (W > 0.0)
                            for (long j = 0; j < V; ++j) r[j] /= W;
                    }
                }
                if (next < 0) {                       /* the extra token from r */
                    double W = 0.0;
                    for (long j = 0; j < V; ++j) W += r[j];
                    if (W > 0.0) {
                        const double mass = u[0] * W;
                        double C = 0.0, Cprev = 0.0;
                        for (long j = 0; j < V; ++j) {
                            Cprev = C;
                            C += r[j];
                            if (C > mass) { extra = j; break; }
                        }
                        if (extra < 0) {
                            for (long j = V - 1; j >= 0; --j)
                                if (r[j] > 0.0) { extra = j; break; }
                            Cprev = W - r[extra];
                            C = W;
                        }
                        const double g1 = C - mass, g0 = mass - Cprev;
                        cdf_gap[b] = (g1 < g0 ? g1 : g0) / W;
                    } else {
                        extra = argmax_first(lp, V);
                    }
                    break;
                }
            }
            pth[depth] = (int32_t)next;
            out[depth] = y[next];
            ++depth;
            node = next;
        }
        out[depth] = (int32_t)extra;
        accepted[b] = (int32_t)depth;
        last_node[b] = (int32_t)node;
    }
    free(lq); free(lp); free(q); free(r);
    return 0;
}
