// ppd_accept.cuh -- device helpers shared by the standalone argmax / acceptance
// kernels and the fused end phase of the attention kernel: the argmax ranking
// rule, the combine of per-split partial maxima, and one warp's exact-matching
// acceptance of one sequence (paper Section 3 steps (2)-(3)).
#pragma once

#include "ppd_device.cuh"
#include "ppd_kernels.h"

#include <climits>

namespace ppd {

// true when (av, ai) ranks before (bv, bi): NaN first (lowest index among
// NaNs), then the larger value, then the lower index.  -0 and +0 compare equal.
PPD_DEV bool ranks_before(float av, int ai, float bv, int bi)
{
    const bool an = av != av, bn = bv != bv;
    if (an || bn) return an && bn ? ai < bi : an;
    if (av != bv) return av > bv;
    return ai < bi;
}

PPD_DEV void consider(float v, int i, float &bv, int &bi)
{
    if (ranks_before(v, i, bv, bi)) {
        bv = v;
        bi = i;
    }
}

// Top-1 index of one row from its `splits` partial (value, index) results.
PPD_DEV int combine_partials(const float *part_val, const int32_t *part_idx, int64_t row, int splits)
{
    float bv = __ldcg(part_val + row * splits);
    int bi = __ldcg(part_idx + row * splits);
    for (int k = 1; k < splits; ++k)
        consider(__ldcg(part_val + row * splits + k), __ldcg(part_idx + row * splits + k), bv, bi);
    return bi;
}

// ------------------------------------------------------------------ softmax statistics
//
// Running statistics of the distribution softmax(x / tau) over a stream of
// logits, kept in base-2 units y = x * k with k = log2(e) / tau:
//   m = max y,  s = sum 2^(y - m),  t = sum 2^(y - m) * (y - m).
// Then lse = ln2 * (m + log2 s) is log sum exp(x / tau) and the entropy is
// H = ln2 * (log2 s - t / s).  A NaN anywhere makes s (and so both) NaN;
// -inf logits contribute nothing.
struct SoftStats {
    float m = -INFINITY, s = 0.f, t = 0.f;
};

// Fold four scaled logits into st.
PPD_DEV void stats_add4(SoftStats &st, float y0, float y1, float y2, float y3)
{
    const float mg = fmaxf(fmaxf(y0, y1), fmaxf(y2, y3));
    if (mg > st.m) {
        if (st.s != 0.f) {
            const float a = ex2(st.m - mg);
            st.t = a * (st.t + (st.m - mg) * st.s);
            st.s *= a;
        }
        st.m = mg;
    }
    const float y[4] = {y0, y1, y2, y3};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float d = y[k] - st.m;
        const float e = (y[k] == -INFINITY) ? 0.f : ex2(d);
        st.s += e;
        st.t += (e > 0.f) ? e * d : ((e == e) ? 0.f : e);
    }
}

// st <- st (+) o.
PPD_DEV void stats_merge(SoftStats &st, const SoftStats &o)
{
    const float M = fmaxf(st.m, o.m);
    float s = 0.f, t = 0.f;
    if (st.s != 0.f) {
        const float a = ex2(st.m - M);
        s += a * st.s;
        t += a * (st.t + (st.m - M) * st.s);
    }
    if (o.s != 0.f) {
        const float a = ex2(o.m - M);
        s += a * o.s;
        t += a * (o.t + (o.m - M) * o.s);
    }
    st.m = M;
    st.s = s;
    st.t = t;
}

// Statistics of one row from its `splits` partial (m, s, t) triples.
PPD_DEV SoftStats combine_stats(const float *part_stats, int64_t row, int splits)
{
    SoftStats st;
    for (int k = 0; k < splits; ++k) {
        const float *ps = part_stats + 3 * (row * splits + k);
        SoftStats o;
        o.m = __ldcg(ps);
        o.s = __ldcg(ps + 1);
        o.t = __ldcg(ps + 2);
        stats_merge(st, o);
    }
    return st;
}

// Natural-log log-sum-exp and entropy from the statistics.
PPD_DEV void stats_finish(const SoftStats &st, float &lse, float &entropy)
{
    const float l2s = __log2f(st.s);
    lse = 0.69314718055994530942f * (st.m + l2s);
    entropy = 0.69314718055994530942f * (l2s - st.t / st.s);
}

struct AcceptResult {
    int n_acc;           // accepted tokens, root included; 0 on error
    int next_token;      // top-1 token at the end node; -1 on error
    int new_prefix_len;  // prefix_len + n_acc (prefix_len on error)
    int status;          // kOk, kErrTree or kErrCapacity
};

// Acceptance of one sequence by one warp (all lanes call it).
//   top     the sequence's T top-1 tokens (node i: the model's prediction after i)
//   pass    pass(i, parent, token): does candidate node i (token >= 0) pass its
//           verification test
//   par,tok the sequence's parent array and candidate token ids (global memory)
//   s_par   kAcceptScratchInts ints of per-warp scratch
//   path    T outputs: accepted nodes in depth order, then -1
// Node 0 is always accepted; node i > 0 when tok[i] >= 0, pass(i, par[i],
// tok[i]) holds and its parent is accepted.  The end node is the deepest
// accepted node, the smallest index among equal depths.  Every lane gets the
// same result.  T <= kMaxTree.
template <class TopLoad, class Pass>
PPD_DEV AcceptResult accept_warp_pass(TopLoad top, Pass pass, const int32_t *par,
                                      const int32_t *tok, int P, int T, int V, int S_max, int lane,
                                      int *s_par, int32_t *path)
{
    uint32_t *s_ok = reinterpret_cast<uint32_t *>(s_par + kMaxTree);
    const int nw = (T + 31) >> 5;
    bool bad = false;
    for (int k = 0; k < nw; ++k) {
        const int i = lane + 32 * k;
        if (i < T) {
            const int pa = __ldg(par + i);
            const int tk = __ldg(tok + i);
            s_par[i] = pa;
            if (i == 0)
                bad |= (pa != -1) || tk < 0 || tk >= V;
            else
                bad |= pa < 0 || pa >= i || tk < -1 || tk >= V;
        }
    }
    __syncwarp();
    bad = __any_sync(0xffffffffu, bad);
    int err = bad ? kErrTree : ((P < 0 || P > S_max) ? kErrCapacity : kOk);

    for (int k = 0; k < nw; ++k) {
        const int i = lane + 32 * k;
        bool ok = false;
        if (i < T && err == kOk) {
            if (i == 0) {
                ok = true;
            } else {
                const int tk = __ldg(tok + i);
                ok = tk >= 0 && pass(i, s_par[i], tk);
            }
        }
        const uint32_t w = __ballot_sync(0xffffffffu, ok);
        if (lane == 0) s_ok[k] = w;
    }
    __syncwarp();

    int best_key = -1;   // (depth << 10) | (1023 - node): deepest, then smallest index
    if (err == kOk) {
        for (int k = 0; k < nw; ++k) {
            const int i = lane + 32 * k;
            if (i < T) {
                int n = i, depth = 0;
                bool good = true;
                while (n > 0) {
                    good &= ((s_ok[n >> 5] >> (n & 31)) & 1u) != 0;
                    n = s_par[n];
                    ++depth;
                }
                if (good) best_key = max(best_key, (depth << 10) | (1023 - i));
            }
        }
    }
    best_key = __reduce_max_sync(0xffffffffu, best_key);
    const int best = 1023 - (best_key & 1023);
    const int n_acc = (best_key >> 10) + 1;
    if (err == kOk && (long long)P + n_acc > S_max) err = kErrCapacity;
    const int n_out = (err == kOk) ? n_acc : 0;

    for (int k = 0; k < nw; ++k) {
        const int i = lane + 32 * k;
        if (i < T && i >= n_out) path[i] = -1;
    }
    if (lane == 0 && err == kOk) {
        int n = best;
        for (int j = n_acc - 1; j >= 0; --j) {
            path[j] = n;
            n = s_par[n];
        }
    }
    AcceptResult r;
    r.n_acc = n_out;
    r.next_token = (err == kOk) ? top(best) : -1;
    r.new_prefix_len = (err == kOk) ? P + n_acc : P;
    r.status = err;
    __syncwarp();
    return r;
}

// ------------------------------------------------------------------ trees of up to 64 nodes
//
// The same acceptance with the tree in registers: node i's values live in lane
// i % 32, slot i / 32, of a two-slot array, and a node's value is fetched with
// two warp shuffles (every lane takes part; n < 64).  No scratch memory: in
// the fused step's side warp, where a round trip to L2 costs about a
// microsecond while the other warps stream K/V, the walk up the tree then
// costs shuffles instead of dependent loads.
template <class V2>
PPD_DEV auto node_value(const V2 (&v)[2], int n) -> V2
{
    const V2 a = __shfl_sync(0xffffffffu, v[0], n & 31);
    const V2 b = __shfl_sync(0xffffffffu, v[1], n & 31);
    return n < 32 ? a : b;
}

// Acceptance of one sequence of T <= 64 nodes by one warp (all lanes call it;
// the rule and the result are those of accept_warp_pass).
//   top    node i's top-1 token in lane i % 32, slot i / 32
//   pass   pass(i, parent, token), called by every lane at once (it may fetch
//          node values); lanes with no node pass parent 0 and token 0
//   path   out: accepted node j (depth order) in lane j % 32, slot j / 32; -1
//          from n_acc on
template <class Pass>
PPD_DEV AcceptResult accept_warp_small(const int (&top)[2], Pass pass, const int32_t *par,
                                       const int32_t *tok, int P, int T, int V, int S_max, int lane,
                                       int (&path)[2])
{
    int pa[2], tk[2];
    bool bad = false;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int i = lane + 32 * k;
        pa[k] = -1;
        tk[k] = -1;
        if (i < T) {
            pa[k] = __ldg(par + i);
            tk[k] = __ldg(tok + i);
            if (i == 0)
                bad |= (pa[k] != -1) || tk[k] < 0 || tk[k] >= V;
            else
                bad |= pa[k] < 0 || pa[k] >= i || tk[k] < -1 || tk[k] >= V;
        }
    }
    bad = __any_sync(0xffffffffu, bad);
    int err = bad ? kErrTree : ((P < 0 || P > S_max) ? kErrCapacity : kOk);

    uint32_t okw[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int i = lane + 32 * k;
        const bool cand = i > 0 && i < T && err == kOk && tk[k] >= 0;
        const bool ps = pass(i, cand ? pa[k] : 0, cand ? tk[k] : 0);
        okw[k] = __ballot_sync(0xffffffffu, (i == 0 && err == kOk) || (cand && ps));
    }

    int best_key = -1;   // (depth << 10) | (1023 - node): deepest, then smallest index
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int i = lane + 32 * k;
        const bool mine = i < T && err == kOk;
        int n = mine ? i : 0, depth = 0;
        bool good = true;
        // a valid tree's parents precede their children: every walk ends at 0
        while (__any_sync(0xffffffffu, n > 0)) {
            const int up = node_value(pa, n);
            if (n > 0) {
                good &= (((n >> 5) ? okw[1] : okw[0]) >> (n & 31) & 1u) != 0;
                n = up;
                ++depth;
            }
        }
        if (mine && good) best_key = max(best_key, (depth << 10) | (1023 - i));
    }
    best_key = __reduce_max_sync(0xffffffffu, best_key);
    const int best = 1023 - (best_key & 1023);
    const int n_acc = (best_key >> 10) + 1;
    if (err == kOk && (long long)P + n_acc > S_max) err = kErrCapacity;
    const int n_out = (err == kOk) ? n_acc : 0;

    path[0] = -1;
    path[1] = -1;
    int n = best;
    for (int j = n_out - 1; j >= 0; --j) {   // warp-uniform trip count
        if (lane == (j & 31)) path[j >> 5 ? 1 : 0] = n;
        n = node_value(pa, n);
    }
    AcceptResult r;
    r.n_acc = n_out;
    const int nt = node_value(top, err == kOk ? best : 0);
    r.next_token = (err == kOk) ? nt : -1;
    r.new_prefix_len = (err == kOk) ? P + n_acc : P;
    r.status = err;
    return r;
}

// Exact matching (Section 3 step (2)): a candidate passes when it equals the
// top-1 token predicted at its parent.
template <class TopLoad>
PPD_DEV AcceptResult accept_warp(TopLoad top, const int32_t *par, const int32_t *tok, int P, int T,
                                 int V, int S_max, int lane, int *s_par, int32_t *path)
{
    return accept_warp_pass(
        top, [&](int, int pa, int tk) { return tk == top(pa); }, par, tok, P, T, V, S_max, lane,
        s_par, path);
}

// Typical acceptance (Section 3 step (2), the second scheme the paper names):
// a candidate t below node j passes when p_t > min(epsilon, delta * exp(-H_j)),
// with p = softmax(logits[j] / tau), from the natural-log log-sum-exp lse[j]
// and entropy ent[j] of that distribution.  `x` is the sequence's logits
// [T][V]; lse / ent load node j's values.
template <class TopLoad, class Lse, class Ent>
PPD_DEV AcceptResult accept_warp_typical(TopLoad top, const float *x, Lse lse, Ent ent,
                                         float inv_temp, float epsilon, float delta,
                                         const int32_t *par, const int32_t *tok, int P, int T,
                                         int V, int S_max, int lane, int *s_par, int32_t *path)
{
    return accept_warp_pass(
        top,
        [&](int, int pa, int tk) {
            const float pt = expf(__ldg(x + (size_t)pa * V + tk) * inv_temp - lse(pa));
            return pt > fminf(epsilon, delta * expf(-ent(pa)));
        },
        par, tok, P, T, V, S_max, lane, s_par, path);
}

// ------------------------------------------------------------------ logits scan

// Top-1 (and with kStats the softmax statistics) of columns [lo, hi) of the
// logits row x by one warp, with kDepth 16-byte loads per lane issued before
// any is used (predicated at the end of the span, so a span of n float4 takes
// ceil(n / (32 kDepth)) round trips); lane 0 holds the result.
template <bool kStats, int kDepth>
PPD_DEV void warp_logit_span(const float *x, int lo, int hi, bool vec, float stat_k, int lane,
                             float &bv, int &bi, SoftStats &st)
{
    bv = -INFINITY;
    bi = INT_MAX;
    st = SoftStats{};
    if (vec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(x);
        const int n4_hi = hi >> 2;
        for (int i = (lo >> 2) + lane; i < n4_hi; i += kDepth * 32) {
            float4 f[kDepth];
#pragma unroll
            for (int k = 0; k < kDepth; ++k)
                if (i + k * 32 < n4_hi) f[k] = __ldcs(x4 + i + k * 32);
#pragma unroll
            for (int k = 0; k < kDepth; ++k) {
                if (i + k * 32 < n4_hi) {
                    const int base = 4 * (i + k * 32);
                    consider(f[k].x, base, bv, bi);
                    consider(f[k].y, base + 1, bv, bi);
                    consider(f[k].z, base + 2, bv, bi);
                    consider(f[k].w, base + 3, bv, bi);
                    if (kStats)
                        stats_add4(st, f[k].x * stat_k, f[k].y * stat_k, f[k].z * stat_k,
                                   f[k].w * stat_k);
                }
            }
        }
    } else {
        for (int i = lo + lane; i < hi; i += kDepth * 32) {
            float v[kDepth];
#pragma unroll
            for (int k = 0; k < kDepth; ++k)
                if (i + k * 32 < hi) v[k] = __ldcs(x + i + k * 32);
#pragma unroll
            for (int k = 0; k < kDepth; ++k) {
                if (i + k * 32 < hi) {
                    consider(v[k], i + k * 32, bv, bi);
                    if (kStats) stats_add4(st, v[k] * stat_k, -INFINITY, -INFINITY, -INFINITY);
                }
            }
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_down_sync(0xffffffffu, bv, off);
        const int oi = __shfl_down_sync(0xffffffffu, bi, off);
        consider(ov, oi, bv, bi);
        if (kStats) {
            SoftStats o;
            o.m = __shfl_down_sync(0xffffffffu, st.m, off);
            o.s = __shfl_down_sync(0xffffffffu, st.s, off);
            o.t = __shfl_down_sync(0xffffffffu, st.t, off);
            stats_merge(st, o);
        }
    }
}

}  // namespace ppd
