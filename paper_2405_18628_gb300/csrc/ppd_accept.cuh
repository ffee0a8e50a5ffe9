// ppd_accept.cuh -- device helpers shared by the standalone argmax / acceptance
// kernels and the fused end phase of the attention kernel: the argmax ranking
// rule, the combine of per-split partial maxima, and one warp's exact-matching
// acceptance of one sequence (paper Section 3 steps (2)-(3)).
#pragma once

#include "ppd_device.cuh"

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

struct AcceptResult {
    int n_acc;           // accepted tokens, root included; 0 on error
    int next_token;      // top-1 token at the end node; -1 on error
    int new_prefix_len;  // prefix_len + n_acc (prefix_len on error)
    int status;          // kOk, kErrTree or kErrCapacity
};

// Exact-matching acceptance of one sequence by one warp (all lanes call it).
//   top     the sequence's T top-1 tokens (node i: the model's prediction after i)
//   par,tok the sequence's parent array and candidate token ids (global memory)
//   s_par   T ints of per-warp shared scratch
//   path    T outputs: accepted nodes in depth order, then -1
// Node 0 is always accepted; node i > 0 when tok[i] >= 0 equals top[par[i]] and
// its parent is accepted.  The end node is the deepest accepted node, the
// smallest index among equal depths.  Every lane gets the same result.
template <class TopLoad>
PPD_DEV AcceptResult accept_warp(TopLoad top, const int32_t *par, const int32_t *tok, int P,
                                 int T, int V, int S_max, int lane, int *s_par, int32_t *path)
{
    bool bad = false;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
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

    uint32_t okw[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = lane + 32 * k;
        bool ok = false;
        if (i < T && err == kOk) {
            if (i == 0) {
                ok = true;
            } else {
                const int tk = __ldg(tok + i);
                ok = tk >= 0 && tk == top(s_par[i]);
            }
        }
        okw[k] = __ballot_sync(0xffffffffu, ok);
    }

    int best_key = -1;   // (depth << 8) | (255 - node): deepest, then smallest index
    if (err == kOk) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int i = lane + 32 * k;
            if (i < T) {
                int n = i, depth = 0;
                bool good = true;
                while (n > 0) {
                    const uint32_t w = (n < 32) ? okw[0] : (n < 64) ? okw[1] : (n < 96) ? okw[2] : okw[3];
                    good &= ((w >> (n & 31)) & 1u) != 0;
                    n = s_par[n];
                    ++depth;
                }
                if (good) best_key = max(best_key, (depth << 8) | (255 - i));
            }
        }
    }
    best_key = __reduce_max_sync(0xffffffffu, best_key);
    const int best = 255 - (best_key & 255);
    const int n_acc = (best_key >> 8) + 1;
    if (err == kOk && (long long)P + n_acc > S_max) err = kErrCapacity;
    const int n_out = (err == kOk) ? n_acc : 0;

#pragma unroll
    for (int k = 0; k < 4; ++k) {
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

}  // namespace ppd
