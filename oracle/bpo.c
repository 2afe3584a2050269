/*
 * BlockPilot reference oracle (fp64, CPU) -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, deliberately unoptimised restatement of what the block-verify
 * hot path of BlockPilot (arxiv 2606.31315) computes.  Only the test-suite, the
 * smoke check and the benchmark's CPU-baseline leg may load this library; the
 * product path never does.  It shares no code, header, table or helper with the
 * CUDA library: every quantity is recomputed here from its definition, in
 * double precision, with the loops in the order the definition states them.
 *
 * Inputs arrive as fp64 arrays that hold the exact values the GPU path sees
 * (bf16 / fp32 values widened without rounding); the LM-head projection takes
 * its bf16 operands as raw bits and widens them itself (the weight has 389 M
 * entries).  Random numbers the method
 * draws (the acceptance uniforms and the resampling uniform) are inputs.
 *
 * Six parts:
 *   bpo_block_attention  -- block attention of a B-token block over a KV cache,
 *                           causal within the block (target verify pass) or
 *                           bidirectional within the block (dLLM drafter pass).
 *   bpo_spec_accept      -- lossless speculative acceptance of a drafted block.
 *   bpo_policy_select    -- the once-per-request block-size predictor.
 *   bpo_lm_head_logits   -- the output projection that turns the final hidden
 *                           states of the verified (and drafted) positions into
 *                           the logits the acceptance reads.
 *   bpo_tau_select       -- Appendix A's model of the expected acceptance length
 *                           tau(b; x) per candidate block size, the optimal size
 *                           B*(x), and the regret of a predicted size.
 *   bpo_verify_commit    -- the step of the decoding loop after acceptance: what
 *                           stays in each sequence's KV cache, and the next block.
 *
 * Readings of the paper where it is silent are documented at each function.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>

#define BPO_OK 0
#define BPO_BAD_ARG 1

#define BPO_MASK_CAUSAL 0
#define BPO_MASK_BIDIR 1

/* ------------------------------------------------------------------------- */
/* Block attention                                                            */
/* ------------------------------------------------------------------------- */
/*
 * Section 2.1 (Problem Formulation) and the Figure 1 caption: the drafter
 * proposes a block of B tokens in one forward pass and the target verifies the
 * whole block in one parallel pass.  The paper does not print the attention
 * itself; this is the standard scaled dot-product attention that both passes
 * run over the KV cache:
 *
 *   O[i, h] = sum_j softmax_j( scale * <q_{i,h}, k_{j, h/g}> + M_ij ) v_{j, h/g}
 *
 * Sequence s owns query rows [cu_q[s], cu_q[s+1]) (its block, B_s rows) and
 * key/value rows [cu_kv[s], cu_kv[s+1]) (its L_s context rows followed by the
 * block's own B_s rows, so kv_len_s = L_s + B_s).  Mask M:
 *   causal (verify):        block query i sees keys 0 .. L_s + i
 *   bidirectional (draft):  every block query sees keys 0 .. L_s + B_s - 1
 * Grouped-query attention: query head h reads KV head h / g, g = Hq / Hkv.
 *
 * Layouts (row-major): q, o [total_q][Hq][D]; k, v [total_kv][Hkv][D];
 * lse [total_q][Hq] (natural-log log-sum-exp of the scaled, masked scores;
 * may be NULL).
 */
int bpo_block_attention(const double *q, const double *k, const double *v,
                        double *o, double *lse, const int32_t *cu_q,
                        const int32_t *cu_kv, int num_seqs, int num_q_heads,
                        int num_kv_heads, int head_dim, int mask, double scale)
{
    if (!q || !k || !v || !o || !cu_q || !cu_kv) return BPO_BAD_ARG;
    if (num_seqs < 0 || num_q_heads < 1 || num_kv_heads < 1 || head_dim < 1)
        return BPO_BAD_ARG;
    if (num_q_heads % num_kv_heads != 0) return BPO_BAD_ARG;
    if (mask != BPO_MASK_CAUSAL && mask != BPO_MASK_BIDIR) return BPO_BAD_ARG;
    for (int s = 0; s < num_seqs; ++s) {
        int nq = cu_q[s + 1] - cu_q[s];
        int nkv = cu_kv[s + 1] - cu_kv[s];
        if (nq < 0 || nkv < nq) return BPO_BAD_ARG;
    }
    const int g = num_q_heads / num_kv_heads;
    const int D = head_dim;
    const int total_q = cu_q[num_seqs];

    /* One independent output row per (query token, query head). */
#pragma omp parallel for schedule(dynamic, 4)
    for (long row = 0; row < (long)total_q * num_q_heads; ++row) {
        const int t = (int)(row / num_q_heads); /* global query index */
        const int h = (int)(row % num_q_heads); /* query head */
        const int kvh = h / g;                  /* its KV head */
        int s = 0;
        while (cu_q[s + 1] <= t) ++s;
        const int B = cu_q[s + 1] - cu_q[s];
        const int i = t - cu_q[s]; /* position inside the block */
        const int kv0 = cu_kv[s];
        const int L = (cu_kv[s + 1] - cu_kv[s]) - B; /* context length */
        const int n_keys = (mask == BPO_MASK_CAUSAL) ? (L + i + 1) : (L + B);

        const double *qr = q + ((size_t)t * num_q_heads + h) * D;
        double *orow = o + ((size_t)t * num_q_heads + h) * D;
        double *sc = (double *)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1));

        /* scores */
        double mx = -INFINITY;
        for (int j = 0; j < n_keys; ++j) {
            const double *kr = k + ((size_t)(kv0 + j) * num_kv_heads + kvh) * D;
            double dot = 0.0;
            for (int d = 0; d < D; ++d) dot += qr[d] * kr[d];
            sc[j] = scale * dot;
            if (sc[j] > mx) mx = sc[j];
        }
        /* softmax by max subtraction */
        double z = 0.0;
        for (int j = 0; j < n_keys; ++j) {
            sc[j] = exp(sc[j] - mx);
            z += sc[j];
        }
        for (int d = 0; d < D; ++d) orow[d] = 0.0;
        for (int j = 0; j < n_keys; ++j) {
            const double *vr = v + ((size_t)(kv0 + j) * num_kv_heads + kvh) * D;
            const double w = sc[j] / z;
            for (int d = 0; d < D; ++d) orow[d] += w * vr[d];
        }
        if (lse) lse[(size_t)t * num_q_heads + h] = mx + log(z);
        free(sc);
    }
    return BPO_OK;
}

/* ------------------------------------------------------------------------- */
/* Lossless speculative acceptance                                            */
/* ------------------------------------------------------------------------- */
/*
 * The paper states the rule only by its properties: the target "accepts the
 * longest consistent prefix" of the drafted block (Figure 1 caption) and the
 * output distribution of the target is preserved exactly (Section 1; Section
 * 3.1, Metrics).  It cites standard speculative sampling for it.  Reading used
 * here (standard speculative sampling applied position by position):
 *
 *   p_i = softmax(target_row_i / T),  q_i = softmax(draft_row_i / T)
 *   a_i = min(1, p_i(x_i) / q_i(x_i))            (x_i = drafted token i)
 *   k   = first i < gamma with u_i >= a_i, else gamma   (accepted prefix)
 *   if k < gamma: emit a token drawn from r = max(0, p_k - q_k) / sum(r)
 *   else:         emit a bonus token drawn from p_gamma
 * The draw is an inverse CDF in vocabulary-index order with the sequence's
 * uniform u_s: the smallest t with C_t > u_s * Z, C_t = sum_{j<=t} r_j,
 * Z = C_{V-1}.  If the residual mass Z is exactly zero (p_k == q_k) the draw is
 * made from p_k instead.  Conventions for the ratio: q(x)=0, p(x)>0 gives 1;
 * both zero gives 0; acceptance is the strict test u_i < a_i with u in [0,1).
 *
 * T == 0 is greedy decoding (Table 2, Temperature = 0): g_i = argmax of
 * target row i (lowest index on ties), accept iff x_i == g_i, emit g_k.
 * Draft logits are not read (and may be NULL) at T == 0.
 *
 * Layout.  Sequence s has gamma_s = cu_draft[s+1] - cu_draft[s] drafted
 * tokens, draft rows [cu_draft[s], cu_draft[s+1]) and gamma_s + 1 target rows
 * starting at cu_draft[s] + s.  out_tokens has the same gamma_s + 1 slots per
 * sequence (starting at cu_draft[s] + s): slots 0..k-1 hold the accepted
 * drafts, slot k the emitted token, the rest -1.  accept_prob [total_draft]
 * holds a_i for every drafted position (evaluated at every position, also
 * those after the first rejection).
 *
 * Diagnostics for comparisons with a lower-precision implementation (both
 * may be NULL):
 *   ratio_margin[s] = min |u_i - a_i| over the positions the test examined
 *                     (0..k, excluding k == gamma), +inf if none;
 *   cdf_margin[s]   = min(u_s*Z - C_{t-1}, C_t - u_s*Z) at the emitted token t,
 *                     in probability mass (the target distribution sums to 1);
 *                     +inf at T == 0.
 */
static void row_softmax(const double *logits, int V, double inv_t, double *p)
{
    double mx = -INFINITY;
    for (int x = 0; x < V; ++x) {
        double z = logits[x] * inv_t;
        if (z > mx) mx = z;
    }
    double sum = 0.0;
    for (int x = 0; x < V; ++x) {
        p[x] = exp(logits[x] * inv_t - mx);
        sum += p[x];
    }
    for (int x = 0; x < V; ++x) p[x] /= sum;
}

static int row_argmax(const double *row, int V)
{
    int best = 0;
    for (int x = 1; x < V; ++x)
        if (row[x] > row[best]) best = x;
    return best;
}

/* Inverse-CDF draw in index order; returns the token and its margin. */
static int inverse_cdf(const double *w, int V, double u, double *margin)
{
    double Z = 0.0;
    for (int x = 0; x < V; ++x) Z += w[x];
    const double thr = u * Z;
    double c = 0.0;
    for (int x = 0; x < V; ++x) {
        double prev = c;
        c += w[x];
        if (c > thr) {
            double m1 = thr - prev, m2 = c - thr;
            *margin = m1 < m2 ? m1 : m2;
            return x;
        }
    }
    /* unreachable for u in [0,1) and Z > 0: C_{V-1} = Z > u*Z */
    *margin = 0.0;
    return V - 1;
}

int bpo_spec_accept(const double *target_logits, const double *draft_logits,
                    const int32_t *draft_tokens, const int32_t *cu_draft,
                    int num_seqs, int vocab, double temperature,
                    const double *u_accept, const double *u_sample,
                    int32_t *n_accepted, int32_t *out_tokens,
                    double *accept_prob, double *ratio_margin,
                    double *cdf_margin)
{
    if (!target_logits || !draft_tokens || !cu_draft || !n_accepted || !out_tokens)
        return BPO_BAD_ARG;
    if (num_seqs < 0 || vocab < 1 || !(temperature >= 0.0)) return BPO_BAD_ARG;
    const int greedy = (temperature == 0.0);
    if (!greedy && (!draft_logits || !u_accept || !u_sample)) return BPO_BAD_ARG;
    for (int s = 0; s < num_seqs; ++s) {
        if (cu_draft[s + 1] < cu_draft[s]) return BPO_BAD_ARG;
        for (int i = cu_draft[s]; i < cu_draft[s + 1]; ++i)
            if (draft_tokens[i] < 0 || draft_tokens[i] >= vocab) return BPO_BAD_ARG;
    }
    const int V = vocab;
    int bad = 0;

#pragma omp parallel for schedule(dynamic, 1)
    for (int s = 0; s < num_seqs; ++s) {
        const int d0 = cu_draft[s];
        const int gamma = cu_draft[s + 1] - d0;
        const int t0 = d0 + s; /* first target row of this sequence */
        const int32_t *x = draft_tokens + d0;
        int32_t *out = out_tokens + t0;
        double rmargin = INFINITY, cmargin = INFINITY;
        int k = gamma;

        if (greedy) {
            for (int i = 0; i < gamma; ++i) {
                int gi = row_argmax(target_logits + (size_t)(t0 + i) * V, V);
                if (accept_prob) accept_prob[d0 + i] = (x[i] == gi) ? 1.0 : 0.0;
            }
            for (int i = 0; i < gamma; ++i) {
                int gi = row_argmax(target_logits + (size_t)(t0 + i) * V, V);
                if (x[i] != gi) { k = i; break; }
            }
            for (int i = 0; i < k; ++i) out[i] = x[i];
            out[k] = row_argmax(target_logits + (size_t)(t0 + k) * V, V);
        } else {
            const double inv_t = 1.0 / temperature;
            double *p = (double *)malloc(sizeof(double) * (size_t)V);
            double *qd = (double *)malloc(sizeof(double) * (size_t)V);
            double *r = (double *)malloc(sizeof(double) * (size_t)V);
            if (!p || !qd || !r) {
                free(p); free(qd); free(r);
#pragma omp atomic write
                bad = 1;
                continue;
            }
            /* ratio a_i at every drafted position */
            double *a = (double *)malloc(sizeof(double) * (size_t)(gamma > 0 ? gamma : 1));
            for (int i = 0; i < gamma; ++i) {
                row_softmax(target_logits + (size_t)(t0 + i) * V, V, inv_t, p);
                row_softmax(draft_logits + (size_t)(d0 + i) * V, V, inv_t, qd);
                const double pp = p[x[i]], qq = qd[x[i]];
                double ai;
                if (qq > 0.0) ai = pp / qq < 1.0 ? pp / qq : 1.0;
                else ai = pp > 0.0 ? 1.0 : 0.0;
                a[i] = ai;
                if (accept_prob) accept_prob[d0 + i] = ai;
            }
            /* longest accepted prefix */
            for (int i = 0; i < gamma; ++i) {
                double m = fabs(u_accept[d0 + i] - a[i]);
                if (m < rmargin) rmargin = m;
                if (!(u_accept[d0 + i] < a[i])) { k = i; break; }
            }
            for (int i = 0; i < k; ++i) out[i] = x[i];
            /* the emitted token */
            row_softmax(target_logits + (size_t)(t0 + k) * V, V, inv_t, p);
            const double *w = p;
            if (k < gamma) {
                row_softmax(draft_logits + (size_t)(d0 + k) * V, V, inv_t, qd);
                double Z = 0.0;
                for (int j = 0; j < V; ++j) {
                    double diff = p[j] - qd[j];
                    r[j] = diff > 0.0 ? diff : 0.0;
                    Z += r[j];
                }
                if (Z > 0.0) w = r;
            }
            out[k] = inverse_cdf(w, V, u_sample[s], &cmargin);
            free(a); free(p); free(qd); free(r);
        }
        for (int i = k + 1; i <= gamma; ++i) out[i] = -1;
        n_accepted[s] = k;
        if (ratio_margin) ratio_margin[s] = rmargin;
        if (cdf_margin) cdf_margin[s] = cmargin;
    }
    return bad ? BPO_BAD_ARG : BPO_OK;
}

/* ------------------------------------------------------------------------- */
/* Block-size policy head                                                     */
/* ------------------------------------------------------------------------- */
/*
 * Section 2.3 (Block Size Predictor) and Section 2.4 (Inference): a small MLP
 * f maps the prefill representation of a request to one logit o_b per
 * candidate block size b, and the block size is B_hat = argmax_b f(.)_b,
 * fixed for the whole request.  Section 3.1 (Implementation Details) fixes two
 * layers with hidden width 2048; the activation is not stated, ReLU is used:
 *
 *   h = max(0, W1 x + b1),  o = W2 h + b2,  B_hat = candidates[argmax_c o_c]
 *
 * (lowest index on ties).  The input is not preprocessed (Table 5: the raw
 * prefill distribution beats softmax or normalisation).  Pooling picks one
 * feature row per request: request n reads row row_index[n] of feats (the
 * last-token row), or row n when row_index is NULL.
 *
 * Layouts: feats rows of d_in values at a stride of row_stride values;
 * w1 [hidden][d_in]; b1 [hidden]; w2 [num_cand][hidden]; b2 [num_cand];
 * logits_out [num_reqs][num_cand] (may be NULL); top2_margin[n] = o_top1 -
 * o_top2 (may be NULL; +inf when num_cand == 1).
 */
int bpo_policy_select(const double *feats, long row_stride,
                      const int32_t *row_index, int num_reqs, int d_in,
                      const double *w1, const double *b1, int hidden,
                      const double *w2, const double *b2, int num_cand,
                      const int32_t *candidates, double *logits_out,
                      int32_t *block_size_out, double *top2_margin)
{
    if (!feats || !w1 || !b1 || !w2 || !b2 || !candidates || !block_size_out)
        return BPO_BAD_ARG;
    if (num_reqs < 0 || d_in < 1 || hidden < 1 || num_cand < 1 || row_stride < d_in)
        return BPO_BAD_ARG;

    for (int n = 0; n < num_reqs; ++n) {
        const long row = row_index ? row_index[n] : n;
        if (row < 0) return BPO_BAD_ARG;
        const double *xr = feats + row * row_stride;
        double *h = (double *)malloc(sizeof(double) * (size_t)hidden);
        double *o = (double *)malloc(sizeof(double) * (size_t)num_cand);
        if (!h || !o) { free(h); free(o); return BPO_BAD_ARG; }
        for (int j = 0; j < hidden; ++j) {
            double acc = b1[j];
            for (int d = 0; d < d_in; ++d) acc += w1[(size_t)j * d_in + d] * xr[d];
            h[j] = acc > 0.0 ? acc : 0.0;
        }
        for (int c = 0; c < num_cand; ++c) {
            double acc = b2[c];
            for (int j = 0; j < hidden; ++j) acc += w2[(size_t)c * hidden + j] * h[j];
            o[c] = acc;
        }
        int best = 0;
        for (int c = 1; c < num_cand; ++c)
            if (o[c] > o[best]) best = c;
        double second = -INFINITY;
        for (int c = 0; c < num_cand; ++c)
            if (c != best && o[c] > second) second = o[c];
        block_size_out[n] = candidates[best];
        if (logits_out)
            for (int c = 0; c < num_cand; ++c) logits_out[(size_t)n * num_cand + c] = o[c];
        if (top2_margin) top2_margin[n] = o[best] - second;
        free(h);
        free(o);
    }
    return BPO_OK;
}

/* ------------------------------------------------------------------------- */
/* LM head: final hidden states -> logits                                     */
/* ------------------------------------------------------------------------- */
/*
 * Section 2.1 and the Figure 1 caption: the target scores every position of
 * the drafted block in one parallel pass, and the acceptance compares its
 * distributions with the drafter's.  The paper does not print the model's
 * output layer; both distributions come from the standard LM head, a linear
 * map of the position's final hidden state h (dimension H) onto the
 * vocabulary:
 *
 *   logits[r][v] = sum_{k < H} W[v][k] * h[r][k]        (v < V)
 *
 * W is [V][H] row-major, h is [rows][H] row-major, both bf16 given as raw
 * bits and widened exactly; the sum is formed in fp64 in index order.
 * abs_dot (may be NULL) receives sum_k |W[v][k] * h[r][k]|, the magnitude
 * that bounds the rounding error of any lower-precision evaluation of the
 * same sum.
 */
static double bf16_bits_to_double(uint16_t b)
{
    union { uint32_t u; float f; } x;
    x.u = (uint32_t)b << 16;
    return (double)x.f;
}

int bpo_lm_head_logits(const uint16_t *w, const uint16_t *h, int rows, int vocab,
                       int hidden, double *logits, double *abs_dot)
{
    if (!w || !h || !logits || rows < 0 || vocab < 1 || hidden < 1) return BPO_BAD_ARG;
    double *hd = (double *)malloc(sizeof(double) * (size_t)(rows > 0 ? rows : 1) * (size_t)hidden);
    if (!hd) return BPO_BAD_ARG;
    for (size_t i = 0; i < (size_t)rows * (size_t)hidden; ++i) hd[i] = bf16_bits_to_double(h[i]);
    int bad = 0;
#pragma omp parallel
    {
        double *wr = (double *)malloc(sizeof(double) * (size_t)hidden);
        if (!wr) {
#pragma omp atomic write
            bad = 1;
        }
#pragma omp for schedule(static)
        for (int v = 0; v < vocab; ++v) {
            if (!wr) continue;
            for (int k = 0; k < hidden; ++k) wr[k] = bf16_bits_to_double(w[(size_t)v * hidden + k]);
            for (int r = 0; r < rows; ++r) {
                const double *hr = hd + (size_t)r * hidden;
                double acc = 0.0, mag = 0.0;
                for (int k = 0; k < hidden; ++k) {
                    acc += wr[k] * hr[k];
                    mag += fabs(wr[k] * hr[k]);
                }
                logits[(size_t)r * vocab + v] = acc;
                if (abs_dot) abs_dot[(size_t)r * vocab + v] = mag;
            }
        }
        free(wr);
    }
    free(hd);
    return bad ? BPO_BAD_ARG : BPO_OK;
}

/* ------------------------------------------------------------------------- */
/* Expected acceptance length per block size (Appendix A)                    */
/* ------------------------------------------------------------------------- */
/*
 * Appendix A.1 writes the expected number of accepted drafts as a sum of
 * prefix-survival probabilities, tau(b; x) = sum_{i=1}^{b} prod_{j=1}^{i}
 * q_j(x, b).  Appendix A.2 factors the conditional acceptance into sample
 * predictability and block-size retention, q_j(x, b) = gamma_j(x) r(b; B) with
 * r(b; B) = exp(-alpha (b - B)^2), so that
 *
 *   tau(b; x) = sum_{i=1}^{b} r(b; B)^i prod_{j=1}^{i} gamma_j(x),
 *
 * and, for a predictability constant over positions (gamma_j = gamma_x), the
 * finite geometric series tau = rho (1 - rho^b) / (1 - rho), rho = gamma_x r.
 * B*(x) = argmax over the candidate set of tau(b; x) (lowest index on ties).
 * Appendix A.3: the regret of a predicted size is R(x) = tau(B*) - tau(B_hat);
 * with L the largest |tau(b1) - tau(b2)| / |b1 - b2| over the candidates
 * (adjacent pairs of the ascending candidate list suffice), R(x) <= L |B* -
 * B_hat|, and so E[R] <= L_tau E|B* - B_hat| with L_tau = max_x L(x).
 *
 * gamma [n][jmax] row-major: gamma_j(x) for j = 1..jmax at column j - 1.  With
 * jmax == 1 the single value is gamma_x and tau uses the geometric form
 * (rho == 1 gives tau = b).  candidates [nc], strictly increasing, each <= jmax
 * unless jmax == 1.  predicted (may be NULL): B_hat per request, one of the
 * candidates.  Outputs: tau [n][nc] (may be NULL), best [n], regret [n] and
 * lips [n] (may be NULL; need predicted for regret), summary[4] (may be NULL):
 * mean regret, mean |B* - B_hat|, L_tau, L_tau * mean |B* - B_hat|.
 */
static double tau_general(const double *g, int b, double r)
{
    double sum = 0.0, prod = 1.0;
    for (int i = 1; i <= b; ++i) {
        prod *= g[i - 1] * r; /* prod_{j<=i} gamma_j r */
        sum += prod;
    }
    return sum;
}

static double tau_geometric(double gx, int b, double r)
{
    const double rho = gx * r;
    if (rho == 1.0) return (double)b;
    return rho * (1.0 - pow(rho, (double)b)) / (1.0 - rho);
}

int bpo_tau_select(const double *gamma, int n, int jmax, const int32_t *cand, int nc,
                   int train_block, double alpha, const int32_t *predicted,
                   double *tau, int32_t *best, double *regret, double *lips,
                   double *summary)
{
    if (!gamma || !cand || !best || n < 0 || jmax < 1 || nc < 1 || !(alpha >= 0.0)) return BPO_BAD_ARG;
    for (int c = 0; c < nc; ++c) {
        if (cand[c] < 1 || (c > 0 && cand[c] <= cand[c - 1])) return BPO_BAD_ARG;
        if (jmax > 1 && cand[c] > jmax) return BPO_BAD_ARG;
    }
    double sum_r = 0.0, sum_d = 0.0, lmax = 0.0;
    for (int x = 0; x < n; ++x) {
        const double *g = gamma + (size_t)x * jmax;
        double t[64];
        if (nc > 64) return BPO_BAD_ARG;
        int bi = 0;
        for (int c = 0; c < nc; ++c) {
            const double d = (double)(cand[c] - train_block);
            const double r = exp(-alpha * d * d);
            t[c] = jmax == 1 ? tau_geometric(g[0], cand[c], r) : tau_general(g, cand[c], r);
            if (tau) tau[(size_t)x * nc + c] = t[c];
            if (t[c] > t[bi]) bi = c;
        }
        best[x] = cand[bi];
        double l = 0.0;
        for (int c = 1; c < nc; ++c) {
            const double s = fabs(t[c] - t[c - 1]) / (double)(cand[c] - cand[c - 1]);
            if (s > l) l = s;
        }
        if (lips) lips[x] = l;
        if (l > lmax) lmax = l;
        if (predicted) {
            int pi = -1;
            for (int c = 0; c < nc; ++c)
                if (cand[c] == predicted[x]) pi = c;
            if (pi < 0) return BPO_BAD_ARG;
            const double rx = t[bi] - t[pi];
            if (regret) regret[x] = rx;
            sum_r += rx;
            sum_d += fabs((double)(cand[bi] - cand[pi]));
        }
    }
    if (summary) {
        summary[0] = n ? sum_r / n : 0.0;
        summary[1] = n ? sum_d / n : 0.0;
        summary[2] = lmax;
        summary[3] = lmax * summary[1];
    }
    return BPO_OK;
}

/* ------------------------------------------------------------------------- */
/* Commit of a verify step (the decoding loop around Figure 1)               */
/* ------------------------------------------------------------------------- */
/*
 * Section 2.1 / Figure 1 and Section 2.4: every step drafts a block of B_s =
 * gamma_s + 1 positions (the anchor -- the last token emitted -- and gamma_s
 * drafts), the target verifies the whole block in one pass (so the K/V rows of
 * all B_s positions are appended to the cache), keeps the longest accepted
 * prefix and emits one more token; the block size is fixed for the request.
 * The rows that stay are those of the anchor and the n_acc accepted drafts:
 *
 *   ctx_s  <-  ctx_s + 1 + n_acc_s         (the rejected drafts' rows drop out)
 *   anchor_s = the token emitted at slot n_acc_s of the step
 *   cu_kv_next[s+1] - cu_kv_next[s] = ctx_s + B_s  (the next verify pass's keys)
 *
 * ctx [S] in/out, n_acc [S], out_tokens [total_draft + S] (slots of sequence s
 * start at cu_draft[s] + s), cu_draft [S+1]; capacity = rows the cache can hold
 * per sequence.  Returns BPO_BAD_ARG (and changes nothing) if some n_acc is
 * outside [0, gamma_s] or the next pass would not fit the capacity.
 */
int bpo_verify_commit(int32_t *ctx, const int32_t *n_acc, const int32_t *out_tokens,
                      const int32_t *cu_draft, int num_seqs, int capacity,
                      int32_t *anchor_out, int32_t *cu_kv_next)
{
    if (!ctx || !n_acc || !out_tokens || !cu_draft || !cu_kv_next || num_seqs < 0) return BPO_BAD_ARG;
    for (int s = 0; s < num_seqs; ++s) {
        const int gamma = cu_draft[s + 1] - cu_draft[s];
        if (n_acc[s] < 0 || n_acc[s] > gamma) return BPO_BAD_ARG;
        if ((long long)ctx[s] + 1 + n_acc[s] + gamma + 1 > capacity) return BPO_BAD_ARG;
    }
    cu_kv_next[0] = 0;
    for (int s = 0; s < num_seqs; ++s) {
        const int gamma = cu_draft[s + 1] - cu_draft[s];
        ctx[s] += 1 + n_acc[s];
        if (anchor_out) anchor_out[s] = out_tokens[cu_draft[s] + s + n_acc[s]];
        cu_kv_next[s + 1] = cu_kv_next[s] + ctx[s] + gamma + 1;
    }
    return BPO_OK;
}

/* Number of OpenMP threads the oracle's parallel loops use (1 without OpenMP). */
#ifdef _OPENMP
#include <omp.h>
int bpo_num_threads(void) { return omp_get_max_threads(); }
/* Sets the thread count of the following parallel loops (n >= 1); no effect on any result. */
void bpo_set_num_threads(int n) { if (n >= 1) omp_set_num_threads(n); }
#else
int bpo_num_threads(void) { return 1; }
void bpo_set_num_threads(int n) { (void)n; }
#endif
