/*
 * ppd_oracle.c -- slow, plain fp64 CPU reference for the verification step of
 * Parallel Prompt Decoding (PPD).
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the test-suite, the smoke check
 * and the benchmark's CPU-baseline / reference arm may load this library.  It
 * shares no source, header, table or helper with the CUDA implementation.
 *
 * Every function is the direct definition of one step, written with plain
 * loops in the paper's order so that it can be checked against the paper by
 * eye.  Floating point is fp64 throughout; inputs stored as bf16 are widened
 * exactly, inputs stored as fp32 are first rounded to bf16 (round to nearest,
 * ties to even) by this file's own bit routine.
 *
 *   oracle_round_bf16      fp32 -> bf16 rounding (IEEE 754 round-half-even)
 *   oracle_tree_attention  tree-masked attention (Section 3 step (1); Section
 *                          4.1: every tree token sees the cached prefix, its
 *                          tree ancestors and itself)
 *   oracle_node_argmax     top-1 token of every tree node's logits (the
 *                          greedy "exact matching" check of Section 3 (2))
 *   oracle_accept_path     longest accepted root-to-node path (Section 3
 *                          steps (2)-(3), exact matching)
 *   oracle_kv_compact      copy the accepted nodes' K/V into the cache
 *                          (Section 3 step (3), "KV cache is updated")
 *   oracle_node_stats      log-sum-exp and entropy of softmax(logits / tau)
 *   oracle_typical_accept  typical acceptance (Section 3 step (2), the
 *                          second verification scheme the paper names)
 *   oracle_topk            the K best tokens of logits rows (ranking order)
 *   oracle_next_tree       next-step candidate tree from the accepted node's
 *                          prompt tokens (Section 3 step (1); Appendix,
 *                          tree states T_k)
 *   oracle_next_tree_ept   the same with the ensemble chains' probabilities
 *                          averaged instead of their logits (the formula of
 *                          Section 3, "Ensemble Prompt Tokens")
 *
 * Status codes (per sequence): 0 ok, 3 malformed tree, 4 capacity / prefix
 * length out of range.  Whole-call argument errors return 1.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum {
    ORC_OK = 0,
    ORC_ERR_INVALID_ARG = 1,
    ORC_ERR_TREE = 3,
    ORC_ERR_CAPACITY = 4
};

/* ------------------------------------------------------------------ bf16 */

/* fp32 -> bf16 with round-to-nearest, ties-to-even on the 16 dropped bits.
 * A carry out of the mantissa correctly bumps the exponent (and the largest
 * finite values round to infinity).  NaN stays NaN (quiet bit forced on). */
static uint16_t round_to_bf16(float x)
{
    uint32_t u;
    memcpy(&u, &x, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u) {
        if (u & 0x007fffffu)
            return (uint16_t)((u >> 16) | 0x0040u);
        return (uint16_t)(u >> 16);
    }
    uint32_t kept = u >> 16;
    uint32_t dropped = u & 0xffffu;
    if (dropped > 0x8000u || (dropped == 0x8000u && (kept & 1u)))
        kept += 1u;
    return (uint16_t)kept;
}

static double bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

void oracle_round_bf16(const float *x, uint16_t *y, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        y[i] = round_to_bf16(x[i]);
}

/* element `idx` of a tensor stored as bf16 (dtype 0) or fp32 (dtype 1),
 * as the bf16 value it denotes, widened to double */
static double load(const void *base, int64_t idx, int dtype)
{
    if (dtype == 0)
        return bf16_to_double(((const uint16_t *)base)[idx]);
    return bf16_to_double(round_to_bf16(((const float *)base)[idx]));
}

/* ------------------------------------------------------------------ trees */

/* A tree is valid when node 0 is the root (parent -1) and every other node's
 * parent precedes it (topological order), so each node has one path to 0. */
static int tree_is_valid(const int32_t *parent, int T)
{
    if (T < 1 || parent[0] != -1)
        return 0;
    for (int i = 1; i < T; ++i)
        if (parent[i] < 0 || parent[i] >= i)
            return 0;
    return 1;
}

/* ------------------------------------------------------------------ attention */

/*
 * Tree-masked attention, one output row per (layer, sequence, head, tree node).
 * Query i of sequence b sees the keys of cache rows 0..P_b-1 and of the tree
 * nodes on its own root path (its ancestors and itself).  With s_j =
 * scale * <q_i, k_j> over those keys: o_i = sum_j exp(s_j - m) v_j /
 * sum_j exp(s_j - m), m = max_j s_j (two passes, fp64).
 *
 * Layouts (row-major): q, k_tree, v_tree [L,B,H,T,D]; k_cache, v_cache
 * [L,B,H,S_max,D]; prefix_len [B]; parent [B,T].  `units` lists which
 * (l*B + b)*H + h slices to compute (NULL: all, in order); out is
 * [n_units,T,D], lse and rowsum (nullable) [n_units,T].  A sequence with a
 * malformed tree or a prefix length outside [0, S_max] gets status 3 / 4 and
 * NaN outputs.
 */
int oracle_tree_attention(const void *q, const void *k_cache, const void *v_cache,
                          const void *k_tree, const void *v_tree, int dtype,
                          const int32_t *prefix_len, const int32_t *parent,
                          int L, int B, int H, int T, int D, int S_max, double scale,
                          const int64_t *units, int64_t n_units,
                          double *out, double *lse, double *rowsum,
                          int32_t *status, int n_threads)
{
    if (L < 1 || B < 1 || H < 1 || T < 1 || D < 1 || S_max < 0 || (dtype != 0 && dtype != 1))
        return ORC_ERR_INVALID_ARG;
    if (scale <= 0.0)
        scale = 1.0 / sqrt((double)D);
    int64_t total = (int64_t)L * B * H;
    if (units == NULL)
        n_units = total;

    int32_t *st = (int32_t *)calloc((size_t)B, sizeof(int32_t));
    for (int b = 0; b < B; ++b) {
        if (!tree_is_valid(parent + (int64_t)b * T, T))
            st[b] = ORC_ERR_TREE;
        else if (prefix_len[b] < 0 || prefix_len[b] > S_max)
            st[b] = ORC_ERR_CAPACITY;
    }
    if (status)
        memcpy(status, st, (size_t)B * sizeof(int32_t));

#ifdef _OPENMP
    if (n_threads > 0)
        omp_set_num_threads(n_threads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int64_t n = 0; n < n_units; ++n) {
        int64_t u = units ? units[n] : n;
        int b = (int)((u / H) % B);
        double *o_unit = out + n * (int64_t)T * D;
        if (u < 0 || u >= total || st[b] != ORC_OK) {
            for (int64_t e = 0; e < (int64_t)T * D; ++e)
                o_unit[e] = NAN;
            for (int i = 0; i < T; ++i) {
                if (lse) lse[n * T + i] = NAN;
                if (rowsum) rowsum[n * T + i] = NAN;
            }
            continue;
        }
        const int32_t *par = parent + (int64_t)b * T;
        int P = prefix_len[b];
        int64_t q_base = u * (int64_t)T * D;          /* [T,D] slice of q / tree K,V */
        int64_t c_base = u * (int64_t)S_max * D;      /* [S_max,D] slice of the cache */
        double *s = (double *)malloc(sizeof(double) * (size_t)(P + T));
        int *key_node = (int *)malloc(sizeof(int) * (size_t)T);

        for (int i = 0; i < T; ++i) {
            /* visible tree keys: walk from node i up to the root */
            int n_tree = 0;
            for (int a = i; a >= 0; a = par[a])
                key_node[n_tree++] = a;

            /* scores */
            int n_keys = P + n_tree;
            for (int j = 0; j < P; ++j) {
                double dot = 0.0;
                for (int d = 0; d < D; ++d)
                    dot += load(q, q_base + (int64_t)i * D + d, dtype) *
                           load(k_cache, c_base + (int64_t)j * D + d, dtype);
                s[j] = scale * dot;
            }
            for (int t = 0; t < n_tree; ++t) {
                double dot = 0.0;
                for (int d = 0; d < D; ++d)
                    dot += load(q, q_base + (int64_t)i * D + d, dtype) *
                           load(k_tree, q_base + (int64_t)key_node[t] * D + d, dtype);
                s[P + t] = scale * dot;
            }

            /* softmax: max, then normaliser */
            double m = -INFINITY;
            for (int j = 0; j < n_keys; ++j)
                if (s[j] > m) m = s[j];
            double denom = 0.0;
            for (int j = 0; j < n_keys; ++j)
                denom += exp(s[j] - m);

            /* weighted sum of the visible value rows */
            double *o = o_unit + (int64_t)i * D;
            for (int d = 0; d < D; ++d)
                o[d] = 0.0;
            double psum = 0.0;
            for (int j = 0; j < n_keys; ++j) {
                double p = exp(s[j] - m) / denom;
                psum += p;
                for (int d = 0; d < D; ++d) {
                    double v = (j < P) ? load(v_cache, c_base + (int64_t)j * D + d, dtype)
                                       : load(v_tree, q_base + (int64_t)key_node[j - P] * D + d, dtype);
                    o[d] += p * v;
                }
            }
            if (lse) lse[n * T + i] = m + log(denom);
            if (rowsum) rowsum[n * T + i] = psum;
        }
        free(s);
        free(key_node);
    }
    free(st);
    return ORC_OK;
}

/* ------------------------------------------------------------------ argmax */

/*
 * Top-1 token of each logits row [rows, V] (fp32): the lowest index holding
 * the maximum.  NaN ranks above every number and the first NaN wins (the
 * convention of numpy.argmax); -0 and +0 compare equal.
 */
void oracle_node_argmax(const float *logits, int64_t rows, int64_t V, int32_t *out)
{
    for (int64_t r = 0; r < rows; ++r) {
        const float *x = logits + r * V;
        int64_t best = 0;
        float best_v = x[0];
        if (!isnan(best_v)) {
            for (int64_t v = 1; v < V; ++v) {
                if (isnan(x[v])) {
                    best = v;
                    break;
                }
                if (x[v] > best_v) {
                    best = v;
                    best_v = x[v];
                }
            }
        }
        out[r] = (int32_t)best;
    }
}

/* ------------------------------------------------------------------ accept */

/*
 * Checks shared by both acceptance rules for one sequence: status 3 for a
 * malformed tree, a root id outside [0, V) or another id outside [-1, V);
 * status 4 for a prefix length outside [0, S_max].
 */
static int check_sequence(const int32_t *par, const int32_t *tok, int T, int V, int P, int S_max)
{
    if (!tree_is_valid(par, T) || tok[0] < 0 || tok[0] >= V)
        return ORC_ERR_TREE;
    for (int i = 1; i < T; ++i)
        if (tok[i] < -1 || tok[i] >= V)
            return ORC_ERR_TREE;
    if (P < 0 || P > S_max)
        return ORC_ERR_CAPACITY;
    return ORC_OK;
}

/*
 * Given ok[i] (node i passes its verification test; ok[0] ignored) for a
 * checked sequence (err == ORC_OK on entry), accept node 0 always and node
 * i > 0 when ok[i] holds and its parent is accepted (recursive definition
 * along the parent pointer).  The end node is the accepted node of greatest
 * depth, the smallest index among equal depths; the path is its root path in
 * depth order, accept_len its length (root included), next_token the top-1
 * token at the end node and new_prefix_len = prefix_len + accept_len.  A path
 * that does not fit in the cache is status 4.  On any error: accept_len 0,
 * path all -1, next_token -1, new_prefix_len = prefix_len.
 */
static int choose_path(const int32_t *par, const int *ok, const int32_t *top, int T, int P,
                       int S_max, int err, int *depth, int *acc, int32_t *pth,
                       int32_t *accept_len, int32_t *next_token, int32_t *new_prefix_len)
{
    int best = 0;
    if (err == ORC_OK) {
        depth[0] = 0;
        acc[0] = 1;
        for (int i = 1; i < T; ++i) {
            int p = par[i];
            depth[i] = depth[p] + 1;
            acc[i] = ok[i] && acc[p];
        }
        for (int i = 1; i < T; ++i)
            if (acc[i] && depth[i] > depth[best])
                best = i;
        if ((int64_t)P + depth[best] + 1 > S_max)
            err = ORC_ERR_CAPACITY;
    }
    for (int i = 0; i < T; ++i)
        pth[i] = -1;
    if (err != ORC_OK) {
        *accept_len = 0;
        *next_token = -1;
        *new_prefix_len = P;
    } else {
        int n = depth[best] + 1;
        int k = n - 1;
        for (int a = best; a >= 0; a = par[a])
            pth[k--] = a;
        *accept_len = n;
        *next_token = top[best];
        *new_prefix_len = P + n;
    }
    return err;
}

/*
 * Exact-matching acceptance of one tree per sequence: node i > 0 passes when
 * it is a candidate token (cand[i] >= 0) equal to the top-1 token predicted at
 * its parent, argmax[parent[i]].  Path choice and errors as in choose_path.
 */
int oracle_accept_path(const int32_t *argmax, const int32_t *cand, const int32_t *parent,
                       const int32_t *prefix_len, int B, int T, int V, int S_max,
                       int32_t *accept_len, int32_t *path, int32_t *next_token,
                       int32_t *new_prefix_len, int32_t *status)
{
    if (B < 1 || T < 1 || V < 1)
        return ORC_ERR_INVALID_ARG;
    int *depth = (int *)malloc(sizeof(int) * (size_t)T);
    int *acc = (int *)malloc(sizeof(int) * (size_t)T);
    int *ok = (int *)malloc(sizeof(int) * (size_t)T);
    for (int b = 0; b < B; ++b) {
        const int32_t *par = parent + (int64_t)b * T;
        const int32_t *tok = cand + (int64_t)b * T;
        const int32_t *top = argmax + (int64_t)b * T;
        int P = prefix_len[b];
        int err = check_sequence(par, tok, T, V, P, S_max);
        ok[0] = 1;
        for (int i = 1; i < T && err == ORC_OK; ++i)
            ok[i] = tok[i] >= 0 && tok[i] == top[par[i]];
        status[b] = choose_path(par, ok, top, T, P, S_max, err, depth, acc, path + (int64_t)b * T,
                                accept_len + b, next_token + b, new_prefix_len + b);
    }
    free(depth);
    free(acc);
    free(ok);
    return ORC_OK;
}

/* ------------------------------------------------------------------ typical acceptance */

/*
 * Statistics of the distribution p = softmax(x / tau) of each logits row
 * [rows, V] (fp32), tau > 0: lse = log sum_v exp(x_v / tau) and the entropy
 * H = -sum_v p_v log p_v, with p_v = exp(x_v / tau - lse).  Written as
 * defined, max-shifted, in fp64; a row holding a NaN gets NaN for both.
 */
void oracle_node_stats(const float *logits, int64_t rows, int64_t V, double tau, double *lse,
                       double *entropy)
{
    for (int64_t r = 0; r < rows; ++r) {
        const float *x = logits + r * V;
        int has_nan = 0;
        double m = -INFINITY;
        for (int64_t v = 0; v < V; ++v) {
            if (isnan(x[v]))
                has_nan = 1;
            else if ((double)x[v] / tau > m)
                m = (double)x[v] / tau;
        }
        if (has_nan) {
            lse[r] = NAN;
            entropy[r] = NAN;
            continue;
        }
        double s = 0.0;
        for (int64_t v = 0; v < V; ++v)
            s += exp((double)x[v] / tau - m);
        double l = m + log(s);
        double h = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double pv = exp((double)x[v] / tau - l);
            if (pv > 0.0)
                h -= pv * ((double)x[v] / tau - l);
        }
        lse[r] = l;
        entropy[r] = h;
    }
}

/*
 * Typical acceptance of one tree per sequence (the paper names it in Section 3
 * step (2) as its second verification scheme and gives no formula; this is
 * the usual form of that rule).  With p = softmax(logits[parent[i]] / tau)
 * and H its entropy, node i > 0 passes when it is a candidate token t =
 * cand[i] >= 0 with
 *     p_t > min(epsilon, delta * exp(-H)).
 * Path choice and errors as in choose_path (next_token is still the top-1
 * token at the end node).  p_tok and threshold [B,T] receive p_t and the
 * right-hand side for every candidate node of a checked sequence and NaN
 * elsewhere.  tau must be positive.
 */
int oracle_typical_accept(const float *logits, const int32_t *argmax, const int32_t *cand,
                          const int32_t *parent, const int32_t *prefix_len, int B, int T, int V,
                          int S_max, double tau, double epsilon, double delta,
                          int32_t *accept_len, int32_t *path, int32_t *next_token,
                          int32_t *new_prefix_len, int32_t *status, double *p_tok,
                          double *threshold)
{
    if (B < 1 || T < 1 || V < 1 || !(tau > 0.0))
        return ORC_ERR_INVALID_ARG;
    int *depth = (int *)malloc(sizeof(int) * (size_t)T);
    int *acc = (int *)malloc(sizeof(int) * (size_t)T);
    int *ok = (int *)malloc(sizeof(int) * (size_t)T);
    double *lse = (double *)malloc(sizeof(double) * (size_t)T);
    double *ent = (double *)malloc(sizeof(double) * (size_t)T);
    for (int b = 0; b < B; ++b) {
        const int32_t *par = parent + (int64_t)b * T;
        const int32_t *tok = cand + (int64_t)b * T;
        const int32_t *top = argmax + (int64_t)b * T;
        const float *x = logits + (int64_t)b * T * V;
        int P = prefix_len[b];
        int err = check_sequence(par, tok, T, V, P, S_max);
        for (int i = 0; i < T; ++i) {
            p_tok[(int64_t)b * T + i] = NAN;
            threshold[(int64_t)b * T + i] = NAN;
        }
        ok[0] = 1;
        if (err == ORC_OK) {
            oracle_node_stats(x, T, V, tau, lse, ent);
            for (int i = 1; i < T; ++i) {
                ok[i] = 0;
                if (tok[i] < 0)
                    continue;
                int p = par[i];
                double pt = exp((double)x[(int64_t)p * V + tok[i]] / tau - lse[p]);
                double th = fmin(epsilon, delta * exp(-ent[p]));
                p_tok[(int64_t)b * T + i] = pt;
                threshold[(int64_t)b * T + i] = th;
                ok[i] = pt > th;
            }
        }
        status[b] = choose_path(par, ok, top, T, P, S_max, err, depth, acc, path + (int64_t)b * T,
                                accept_len + b, next_token + b, new_prefix_len + b);
    }
    free(depth);
    free(acc);
    free(ok);
    free(lse);
    free(ent);
    return ORC_OK;
}

/* ------------------------------------------------------------------ next-step candidates */

/* Ranking of tokens by logit: a NaN before any number (the lower index first
 * among NaNs), then the larger value, then the lower index -- the argmax rule
 * extended to an order. */
static int ranks_before(float av, int64_t ai, float bv, int64_t bi)
{
    int an = isnan(av), bn = isnan(bv);
    if (an || bn)
        return an && bn ? ai < bi : an;
    if (av != bv)
        return av > bv;
    return ai < bi;
}

/*
 * The K best tokens of each logits row [rows, V] in ranking order, out
 * [rows][K], by repeated selection of the best token not yet taken.
 * Requires 1 <= K <= V.
 */
void oracle_topk(const float *logits, int64_t rows, int64_t V, int K, int32_t *out)
{
    char *taken = (char *)malloc((size_t)V);
    for (int64_t r = 0; r < rows; ++r) {
        const float *x = logits + r * V;
        memset(taken, 0, (size_t)V);
        for (int k = 0; k < K; ++k) {
            int64_t best = -1;
            for (int64_t v = 0; v < V; ++v)
                if (!taken[v] && (best < 0 || ranks_before(x[v], v, x[best], best)))
                    best = v;
            taken[best] = 1;
            out[r * K + k] = (int32_t)best;
        }
    }
    free(taken);
}

/* The K best of x[0..V) in ranking order (NaN first, then larger, then lower index). */
static int ranks_before_d(double av, int64_t ai, double bv, int64_t bi)
{
    int an = isnan(av), bn = isnan(bv);
    if (an || bn)
        return an && bn ? ai < bi : an;
    if (av != bv)
        return av > bv;
    return ai < bi;
}

static void topk_d(const double *x, int64_t V, int K, int32_t *out, char *taken)
{
    memset(taken, 0, (size_t)V);
    for (int k = 0; k < K; ++k) {
        int64_t best = -1;
        for (int64_t v = 0; v < V; ++v)
            if (!taken[v] && (best < 0 || ranks_before_d(x[v], v, x[best], best)))
                best = v;
        taken[best] = 1;
        out[k] = (int32_t)best;
    }
}

/* ln sum_v exp(x[v]) in fp64, shifted by the row's maximum: NaN if the row
 * holds a NaN, or if its maximum is +inf or -inf (so every probability of
 * such a row is NaN). */
static double row_lse(const float *x, int64_t V)
{
    double m = -INFINITY;
    int nan_seen = 0;
    for (int64_t v = 0; v < V; ++v) {
        if (isnan(x[v]))
            nan_seen = 1;
        else if ((double)x[v] > m)
            m = (double)x[v];
    }
    if (nan_seen)
        return NAN;
    double sum = 0.0;
    for (int64_t v = 0; v < V; ++v)
        sum += exp((double)x[v] - m);
    return m + log(sum);
}

/*
 * Next-step candidate tree of each sequence (Section 3 step (1): the prompt
 * tokens appended to a guess token predict the tokens after it; Appendix,
 * Definition of tree states: a tree exists in states T_k whose candidate
 * subtree has depth at most k, k being set by the prompt tokens available).
 *
 * e = path[b][accept_len[b] - 1] is the accepted end node.  With n_ept
 * ensemble prompt tokens (Section 3, "Ensemble Prompt Tokens": every prompt
 * token position holds n_ept tokens, each seeing only its own chain, and the
 * guess comes from the average of their logits): the first n_ept children of
 * e with cand_tokens -1, in index order, head n_ept chains, each continued by
 * the lowest-index such child of its last node; k = the shortest chain's
 * length (0 if e has fewer than n_ept prompt children), capped at
 * n_states - 1.  The logits for depth d are those of the chains' nodes at
 * position d averaged in fp32 -- summed in chain order, then divided by
 * n_ept -- and their K best tokens (oracle_topk order) are the guesses for
 * depth d of the next tree.  n_ept = 1 is a single chain and plain logits.  Template state k: tmpl_parent[k][i] (node 0
 * the root, parent -1) and tmpl_rank[k][i] (rank r >= 0: a candidate node, -1:
 * a prompt node; ignored for the root).  Outputs: next_parent[b] =
 * tmpl_parent[k]; next_cand[b][0] = next_token[b]; a candidate node at
 * candidate depth d (candidate nodes on its path, root excluded) gets guess r
 * of depth d; prompt nodes get -1; next_state[b] = k.  Status 3 (and outputs
 * all -1, next_state -1) when accept_len[b] < 1, next_token[b] < 0, or
 * template k is not a tree in topological order, has a candidate below a
 * prompt node, a candidate deeper than k, or a rank outside [0, K).
 */
/*
 * ept_mean = 1 (oracle_next_tree_ept): with n_ept > 1 the guesses for depth d
 * are instead the K best tokens of the mean of the chains' probabilities at
 * position d, p(v) = (1/n_ept) sum_j exp(x_j[v] - lse_j), lse_j = ln sum_v
 * exp(x_j[v]), all in fp64 (row_lse: a chain row holding a NaN or a +-inf
 * maximum makes every p NaN); ranked like the logits (NaN first, then larger,
 * then lower index).  n_ept = 1 ranks the plain logits, which order the
 * tokens as their probabilities do.  ept_mean = 0 is oracle_next_tree.
 */
int oracle_next_tree_ept(const float *logits, const int32_t *parent, const int32_t *cand,
                         const int32_t *path, const int32_t *accept_len, const int32_t *next_token,
                         int B, int T, int V, int n_states, int T_next, const int32_t *tmpl_parent,
                         const int32_t *tmpl_rank, int K, int n_ept, int ept_mean,
                         int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                         int32_t *status)
{
    if (B < 1 || T < 1 || V < 1 || n_states < 1 || T_next < 1 || K < 1 || K > V || n_ept < 1 ||
        ept_mean < 0 || ept_mean > 1)
        return ORC_ERR_INVALID_ARG;
    double *pmean = (double *)malloc(sizeof(double) * (size_t)V);
    double *lse = (double *)malloc(sizeof(double) * (size_t)n_ept);
    char *taken = (char *)malloc((size_t)V);
    int32_t *top = (int32_t *)malloc(sizeof(int32_t) * (size_t)K);
    int *cdepth = (int *)malloc(sizeof(int) * (size_t)T_next);
    int *chain = (int *)malloc(sizeof(int) * (size_t)(T + 1) * (size_t)n_ept);
    float *avg = (float *)malloc(sizeof(float) * (size_t)V);
    for (int b = 0; b < B; ++b) {
        const int32_t *par = parent + (int64_t)b * T;
        const int32_t *tok = cand + (int64_t)b * T;
        int32_t *np = next_parent + (int64_t)b * T_next;
        int32_t *nc = next_cand + (int64_t)b * T_next;
        int err = ORC_OK, k = 0;
        int n = accept_len[b];
        if (n < 1 || n > T || next_token[b] < 0)
            err = ORC_ERR_TREE;
        if (err == ORC_OK) {
            int e = path[(int64_t)b * T + n - 1];
            /* the n_ept prompt chains below the end node: chain[j * (T + 1) + d] */
            int heads = 0;
            for (int i = e + 1; i < T && heads < n_ept; ++i)
                if (par[i] == e && tok[i] == -1)
                    chain[(int64_t)(heads++) * (T + 1)] = i;
            if (heads < n_ept) {
                k = 0;
            } else {
                k = T;
                for (int j = 0; j < n_ept; ++j) {
                    int *cj = chain + (int64_t)j * (T + 1);
                    int len = 1, cur = cj[0];
                    while (1) {
                        int nxt = -1;
                        for (int i = cur + 1; i < T; ++i)
                            if (par[i] == cur && tok[i] == -1) {
                                nxt = i;
                                break;
                            }
                        if (nxt < 0)
                            break;
                        cj[len++] = nxt;
                        cur = nxt;
                    }
                    if (len < k)
                        k = len;
                }
            }
            if (k > n_states - 1)
                k = n_states - 1;
            /* template k */
            const int32_t *tp = tmpl_parent + (int64_t)k * T_next;
            const int32_t *tr = tmpl_rank + (int64_t)k * T_next;
            if (!tree_is_valid(tp, T_next))
                err = ORC_ERR_TREE;
            for (int i = 1; i < T_next && err == ORC_OK; ++i) {
                int p = tp[i];
                if (tr[i] >= 0) {
                    if (p > 0 && tr[p] < 0)
                        err = ORC_ERR_TREE;          /* a candidate below a prompt node */
                    cdepth[i] = (p == 0 ? 0 : cdepth[p]) + 1;
                    if (cdepth[i] > k || tr[i] >= K)
                        err = ORC_ERR_TREE;
                } else {
                    cdepth[i] = -1;
                }
            }
            if (err == ORC_OK) {
                for (int i = 0; i < T_next; ++i) {
                    np[i] = tp[i];
                    nc[i] = -1;
                }
                nc[0] = next_token[b];
                for (int d = 1; d <= k; ++d) {
                    if (ept_mean == 1 && n_ept > 1) {
                        /* the chains' probabilities at position d, averaged */
                        for (int j = 0; j < n_ept; ++j)
                            lse[j] = row_lse(logits + ((int64_t)b * T + chain[(int64_t)j * (T + 1) + d - 1]) * V, V);
                        for (int64_t v = 0; v < V; ++v) {
                            double sum = 0.0;
                            for (int j = 0; j < n_ept; ++j)
                                sum += exp((double)logits[((int64_t)b * T + chain[(int64_t)j * (T + 1) + d - 1]) * V + v] - lse[j]);
                            pmean[v] = sum / (double)n_ept;
                        }
                        topk_d(pmean, V, K, top, taken);
                    } else {
                        for (int64_t v = 0; v < V; ++v) {
                            float sum = logits[((int64_t)b * T + chain[d - 1]) * V + v];
                            for (int j = 1; j < n_ept; ++j)
                                sum += logits[((int64_t)b * T + chain[(int64_t)j * (T + 1) + d - 1]) * V + v];
                            avg[v] = sum / (float)n_ept;
                        }
                        oracle_topk(avg, 1, V, K, top);
                    }
                    for (int i = 1; i < T_next; ++i)
                        if (tr[i] >= 0 && cdepth[i] == d)
                            nc[i] = top[tr[i]];
                }
                next_state[b] = k;
            }
        }
        if (err != ORC_OK) {
            for (int i = 0; i < T_next; ++i) {
                np[i] = -1;
                nc[i] = -1;
            }
            next_state[b] = -1;
        }
        status[b] = err;
    }
    free(top);
    free(cdepth);
    free(chain);
    free(avg);
    free(pmean);
    free(lse);
    free(taken);
    return ORC_OK;
}

int oracle_next_tree(const float *logits, const int32_t *parent, const int32_t *cand,
                     const int32_t *path, const int32_t *accept_len, const int32_t *next_token,
                     int B, int T, int V, int n_states, int T_next, const int32_t *tmpl_parent,
                     const int32_t *tmpl_rank, int K, int n_ept, int32_t *next_parent,
                     int32_t *next_cand, int32_t *next_state, int32_t *status)
{
    return oracle_next_tree_ept(logits, parent, cand, path, accept_len, next_token, B, T, V,
                                n_states, T_next, tmpl_parent, tmpl_rank, K, n_ept, 0, next_parent,
                                next_cand, next_state, status);
}

/* ------------------------------------------------------------------ compaction */

/*
 * For every (layer, sequence, head): cache row prefix_len[b] + j <- tree row
 * path[b][j] for j < accept_len[b], for K and V.  Rows are copied as raw bytes
 * (elem_bytes per element).  Every other cache row is left untouched.
 * Sequences whose accept_len is 0 are skipped; a path entry outside [0, T) or
 * a destination beyond S_max makes the call return 1 without copying that row.
 */
int oracle_kv_compact(void *k_cache, void *v_cache, const void *k_tree, const void *v_tree,
                      const int32_t *path, const int32_t *accept_len, const int32_t *prefix_len,
                      int L, int B, int H, int T, int D, int S_max, int elem_bytes)
{
    int rc = ORC_OK;
    size_t row = (size_t)D * (size_t)elem_bytes;
    for (int l = 0; l < L; ++l)
        for (int b = 0; b < B; ++b)
            for (int h = 0; h < H; ++h) {
                int64_t u = ((int64_t)l * B + b) * H + h;
                int n = accept_len[b];
                for (int j = 0; j < n; ++j) {
                    int src = path[(int64_t)b * T + j];
                    int64_t dst = (int64_t)prefix_len[b] + j;
                    if (src < 0 || src >= T || dst < 0 || dst >= S_max) {
                        rc = ORC_ERR_INVALID_ARG;
                        continue;
                    }
                    memcpy((char *)k_cache + ((u * S_max + dst) * (int64_t)row),
                           (const char *)k_tree + ((u * T + src) * (int64_t)row), row);
                    memcpy((char *)v_cache + ((u * S_max + dst) * (int64_t)row),
                           (const char *)v_tree + ((u * T + src) * (int64_t)row), row);
                }
            }
    return rc;
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
