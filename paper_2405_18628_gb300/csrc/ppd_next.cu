// ppd_next.cu -- next-step candidate tree of the PPD decode loop (paper
// Section 3 step (1): the prompt tokens appended to a guess token predict the
// tokens that follow it; Section 3, Ensemble Prompt Tokens: each prompt
// position holds n_ept tokens, the j-th seeing only the j-th of the positions
// before it, and the guess comes from the average of their logits -- or, in
// the formula the section gives, of their probabilities; Appendix,
// Definition of tree states: the next tree takes state T_k, whose candidate
// subtree is at most k deep, k being the number of prompt positions left
// below the accepted token).
//
// Kernel 1, one block per (sequence, chain position d): finds the n_ept
// prompt chains below the accepted end node (warp ballots over the parent
// array, one warp per chain) and, if d is within the state, the K best tokens
// of the chains' averaged logits (or probabilities) at position d -- every
// thread keeps its own top-K over a strided slice of the row, then K rounds of
// a block-wide best-of-heads merge.  The probability mode first takes each
// chain row's log-sum-exp (one warp a row, an online maximum and sum), then
// ranks sum_j exp(x_j - lse_j): the mean without its 1/n_ept, which no
// ranking sees.  Kernel 2, one warp per sequence: fills the state's
// template with the root token and the guesses.
#include "ppd.h"
#include "ppd_accept.cuh"
#include "ppd_device.cuh"
#include "ppd_kernels.h"

#include <climits>

namespace ppd {

// The lowest-index child i > cur of node cur with cand -1 (a prompt token), or
// -1; one warp, the result is warp-uniform.
PPD_DEV int next_prompt_child(const int32_t *par, const int32_t *tok, int T, int cur, int lane)
{
    for (int i0 = (cur + 1) & ~31; i0 < T; i0 += 32) {
        const int i = i0 + lane;
        const bool hit = i < T && i > cur && __ldg(par + i) == cur && __ldg(tok + i) == -1;
        const unsigned m = __ballot_sync(0xffffffffu, hit);
        if (m) return i0 + __ffs(m) - 1;
    }
    return -1;
}

// ln sum_v exp(x[v]) of one row, by one warp: NaN if the row holds a NaN or
// +inf, or if every entry is -inf (each probability of such a row is NaN).
// -inf entries add nothing; every exponent is a difference <= 0, so nothing
// overflows.
PPD_DEV float row_lse_warp(const float *x, int V, int lane)
{
    constexpr float kLog2e = 1.4426950408889634f;
    float m = -INFINITY, s = 0.f;
    bool bad = false;
    for (int v = lane; v < V; v += 32) {
        const float xv = __ldg(x + v);
        if (isnan(xv) || xv == INFINITY) {
            bad = true;
        } else if (xv > m) {
            s = s * exp2f((m - xv) * kLog2e) + 1.f;
            m = xv;
        } else if (xv > -INFINITY) {
            s += exp2f((xv - m) * kLog2e);
        }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, off);
        const float os = __shfl_xor_sync(0xffffffffu, s, off);
        const float nm = fmaxf(m, om);
        if (nm > -INFINITY)
            s = (m > -INFINITY ? s * exp2f((m - nm) * kLog2e) : 0.f) +
                (om > -INFINITY ? os * exp2f((om - nm) * kLog2e) : 0.f);
        m = nm;
    }
    bad = __any_sync(0xffffffffu, bad);
    return (bad || m == -INFINITY) ? NAN : m + logf(s);
}

// Top-K (K <= kNextMaxK) of the averaged logits (ept_mean 0) or probabilities
// (ept_mean 1) at chain position d (1-based) of sequence b, written to
// topk[(b * (n_states - 1) + d - 1) * K ...] in ranking order (NaN first, then
// larger value, then lower index).  The blocks of position 1 also write the
// state k of their sequence to kstate[b].
__global__ void __launch_bounds__(256)
next_topk_kernel(const float *__restrict__ logits, const int32_t *parent, const int32_t *cand,
                 const int32_t *path, const int32_t *accept_len, int T, int V, int n_states, int K,
                 int n_ept, int ept_mean, int32_t *topk, int32_t *kstate)
{
    constexpr float kLog2e = 1.4426950408889634f;
    __shared__ int s_head[kNextMaxEpt];
    __shared__ float s_lse[kNextMaxEpt];
    __shared__ int s_len[kNextMaxEpt];
    __shared__ int s_node[kNextMaxEpt];
    __shared__ int s_nh, s_k;
    __shared__ float s_v[8];
    __shared__ int s_i[8], s_t[8];
    __shared__ int s_win;
    const int b = blockIdx.x;
    const int d = blockIdx.y + 1;
    const int cap = n_states - 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t *par = parent + (size_t)b * T;
    const int32_t *tok = cand + (size_t)b * T;
    // the chain heads: the first n_ept prompt children of the end node
    if (warp == 0) {
        int cnt = 0;
        const int n = __ldg(accept_len + b);
        const int e = (n >= 1 && n <= T) ? __ldg(path + (size_t)b * T + n - 1) : -1;
        if (e >= 0 && e < T) {
            for (int i0 = (e + 1) & ~31; i0 < T && cnt < n_ept; i0 += 32) {
                const int i = i0 + lane;
                const bool hit = i < T && i > e && __ldg(par + i) == e && __ldg(tok + i) == -1;
                const unsigned m = __ballot_sync(0xffffffffu, hit);
                const int pos = cnt + __popc(m & ((1u << lane) - 1u));
                if (hit && pos < n_ept) s_head[pos] = i;
                cnt += __popc(m);
            }
        }
        if (lane == 0) s_nh = min(cnt, n_ept);
    }
    __syncthreads();
    // each chain's length (capped) and its node at position d, one warp a chain
    if (s_nh == n_ept) {
        for (int j = warp; j < n_ept; j += 8) {
            int cur = s_head[j], len = 1, node = d == 1 ? cur : -1;
            while (len < cap) {
                const int nxt = next_prompt_child(par, tok, T, cur, lane);
                if (nxt < 0) break;
                cur = nxt;
                ++len;
                if (len == d) node = cur;
            }
            if (lane == 0) {
                s_len[j] = len;
                s_node[j] = node;
            }
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int k = 0;
        if (s_nh == n_ept) {
            k = cap;
            for (int j = 0; j < n_ept; ++j) k = min(k, s_len[j]);
        }
        s_k = k;
        if (d == 1) kstate[b] = k;
    }
    __syncthreads();
    if (d > s_k) return;   // uniform over the block
    const float *x0 = logits + ((size_t)b * T + s_node[0]) * V;
    const float n_f = (float)n_ept;
    const bool probs = ept_mean == 1 && n_ept > 1;
    if (probs) {
        for (int j = warp; j < n_ept; j += 8) {
            const float l = row_lse_warp(logits + ((size_t)b * T + s_node[j]) * V, V, lane);
            if (lane == 0) s_lse[j] = l;
        }
        __syncthreads();
    }

    // this thread's best K over its slice, best first
    float hv[kNextMaxK];
    int hi[kNextMaxK];
#pragma unroll
    for (int r = 0; r < kNextMaxK; ++r) {
        hv[r] = -INFINITY;
        hi[r] = INT_MAX;
    }
    float tv = -INFINITY;   // the K-th best so far (the entry a new token must beat)
    int ti = INT_MAX;
    for (int v = threadIdx.x; v < V; v += 256) {
        float xv;
        if (probs) {
            // sum_j p_j(v), chain order; a NaN lse_j makes every score NaN
            xv = 0.f;
            for (int j = 0; j < n_ept; ++j)
                xv += exp2f((__ldcs(logits + ((size_t)b * T + s_node[j]) * V + v) - s_lse[j]) * kLog2e);
        } else if (n_ept > 1) {
            xv = __ldcs(x0 + v);
            // the EPT average: summed in chain order, then one IEEE division
            for (int j = 1; j < n_ept; ++j) xv += __ldcs(logits + ((size_t)b * T + s_node[j]) * V + v);
            xv = xv / n_f;
        } else {
            xv = __ldcs(x0 + v);
        }
        if (!ranks_before(xv, v, tv, ti)) continue;
        // insert, shifting worse entries down (slots K.. stay unused)
        float cv = xv;
        int ci = v;
#pragma unroll
        for (int r = 0; r < kNextMaxK; ++r) {
            if (r < K && ranks_before(cv, ci, hv[r], hi[r])) {
                const float sv = hv[r];
                const int si = hi[r];
                hv[r] = cv;
                hi[r] = ci;
                cv = sv;
                ci = si;
            }
        }
#pragma unroll
        for (int r = 0; r < kNextMaxK; ++r)
            if (r == K - 1) {
                tv = hv[r];
                ti = hi[r];
            }
    }

    // K rounds: the best head over the block is the next token; its owner pops it
    for (int r = 0; r < K; ++r) {
        float bv = hv[0];
        int bi = hi[0], bt = threadIdx.x;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            const int ot = __shfl_xor_sync(0xffffffffu, bt, off);
            if (ranks_before(ov, oi, bv, bi)) {
                bv = ov;
                bi = oi;
                bt = ot;
            }
        }
        if (lane == 0) {
            s_v[warp] = bv;
            s_i[warp] = bi;
            s_t[warp] = bt;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            for (int w = 1; w < 8; ++w)
                if (ranks_before(s_v[w], s_i[w], bv, bi)) {
                    bv = s_v[w];
                    bi = s_i[w];
                    bt = s_t[w];
                }
            topk[((size_t)b * (n_states - 1) + d - 1) * K + r] = bi;
            s_win = bt;
        }
        __syncthreads();
        if ((int)threadIdx.x == s_win) {
#pragma unroll
            for (int q = 0; q + 1 < kNextMaxK; ++q) {
                hv[q] = hv[q + 1];
                hi[q] = hi[q + 1];
            }
            hv[kNextMaxK - 1] = -INFINITY;
            hi[kNextMaxK - 1] = INT_MAX;
        }
        __syncthreads();
    }
}

// One warp per sequence: state, template checks, and the next tree.
__global__ void __launch_bounds__(128)
next_assemble_kernel(const int32_t *parent, const int32_t *cand, const int32_t *path,
                     const int32_t *accept_len, const int32_t *next_token, int B, int T,
                     int n_states, int T_next, const int32_t *tmpl_parent, const int32_t *tmpl_rank,
                     int K, const int32_t *topk, const int32_t *kstate, int32_t *next_parent,
                     int32_t *next_cand, int32_t *next_state, int32_t *status)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.x * 4 + warp;
    if (b >= B) return;
    const int n = __ldg(accept_len + b);
    const int nt = __ldg(next_token + b);
    bool bad = !(n >= 1 && n <= T && nt >= 0);
    int k = 0;
    if (!bad) {
        const int e = __ldg(path + (size_t)b * T + n - 1);
        bad = !(e >= 0 && e < T);
        if (!bad && n_states > 1) k = __ldg(kstate + b);
    }
    const int32_t *tp = tmpl_parent + (size_t)k * T_next;
    const int32_t *tr = tmpl_rank + (size_t)k * T_next;
    int32_t *np = next_parent + (size_t)b * T_next;
    int32_t *nc = next_cand + (size_t)b * T_next;
    // template checks and each node's candidate depth (walk to the root)
    for (int i = lane; i < T_next && !bad; i += 32) {
        const int pi = __ldg(tp + i);
        if (i == 0) {
            bad |= pi != -1;
            continue;
        }
        bad |= pi < 0 || pi >= i;
        const int r = __ldg(tr + i);
        if (r >= 0) bad |= r >= K;
    }
    bad = __any_sync(0xffffffffu, bad);
    if (!bad) {
        for (int i = lane; i < T_next; i += 32) {
            const int r = __ldg(tr + i);
            int tokv = -1;
            if (i == 0) {
                tokv = nt;
            } else if (r >= 0) {
                int depth = 0, a = i;
                bool ok = true;
                while (a > 0) {
                    ok &= __ldg(tr + a) >= 0;     // every node above a candidate is a candidate
                    ++depth;
                    a = __ldg(tp + a);
                }
                if (!ok || depth > k) {
                    tokv = INT_MIN;               // marks a bad template
                } else {
                    tokv = __ldg(topk + ((size_t)b * (n_states - 1) + depth - 1) * K + r);
                }
            }
            nc[i] = tokv;
            np[i] = __ldg(tp + i);
        }
        __syncwarp();
        bool inv = false;
        for (int i = lane; i < T_next; i += 32) inv |= nc[i] == INT_MIN;
        bad = __any_sync(0xffffffffu, inv);
    }
    if (bad) {
        for (int i = lane; i < T_next; i += 32) {
            np[i] = -1;
            nc[i] = -1;
        }
    }
    if (lane == 0) {
        next_state[b] = bad ? -1 : k;
        status[b] = bad ? kErrTree : kOk;
    }
}

cudaError_t launch_next_tree(const float *logits, const int32_t *parent, const int32_t *cand,
                             const int32_t *path, const int32_t *accept_len,
                             const int32_t *next_token, int B, int T, int V, int n_states,
                             int T_next, const int32_t *tmpl_parent, const int32_t *tmpl_rank, int K,
                             int n_ept, int ept_mean, int32_t *topk, int32_t *kstate,
                             int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                             int32_t *status, cudaStream_t stream)
{
    if (n_states > 1) {
        next_topk_kernel<<<dim3((unsigned)B, (unsigned)(n_states - 1)), 256, 0, stream>>>(
            logits, parent, cand, path, accept_len, T, V, n_states, K, n_ept, ept_mean, topk,
            kstate);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    next_assemble_kernel<<<(B + 3) / 4, 128, 0, stream>>>(parent, cand, path, accept_len, next_token,
                                                          B, T, n_states, T_next, tmpl_parent,
                                                          tmpl_rank, K, topk, kstate,
                                                          next_parent, next_cand, next_state,
                                                          status);
    return cudaGetLastError();
}

}  // namespace ppd
