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
// The log-sum-exp and top-K kernels first find, per (sequence, chain position
// d), the n_ept prompt chains below the accepted end node (find_chains: each node's
// lowest-index prompt child by a shared-memory minimum, one node per thread;
// the end node's prompt children ranked by ballots; each chain walked through
// those links).  The probability mode then takes each chain row's log-sum-exp
// (next_lse_kernel, one block a row).  next_topk_kernel shares each row's
// columns among up to kNextMaxSplit blocks: every thread keeps its own top-K
// of the averaged logits (or of sum_j exp(x_j - lse_j), the probability mean
// without its 1/n_ept, which no ranking sees) over a strided slice of its
// block's columns, read four 16-byte loads per row at a time; each warp takes
// the best K of its lanes (K rounds of a shuffle maximum, the winning lane
// popping its head) and one warp the best K of the warps, a partial list.
// next_topk_merge_kernel, one warp per (sequence, position), takes the best K
// of the partial lists, and next_assemble_kernel, one warp per sequence, fills
// the state's template with the root token and the guesses.
#include "ppd.h"
#include "ppd_accept.cuh"
#include "ppd_device.cuh"
#include "ppd_kernels.h"

#include <climits>

namespace ppd {

constexpr int kTopkThreads = 512;                  // one tree node per thread (T <= 512)
constexpr int kTopkWarps = kTopkThreads / 32;
constexpr int kBatch = 4;                          // 16-byte loads in flight per row and thread
constexpr float kLog2e = 1.4426950408889634f;
static_assert(kMaxTree <= kTopkThreads, "find_chains takes one tree node per thread");

// The kernels of one call form a chain of programmatic launches: each lets
// the next one launch at its entry, and the next does its setup from the
// call's inputs (the chains, the template) before it waits for the previous
// grid to complete and reads what that grid wrote.  The first kernel of a
// call is launched in plain stream order, so the call's inputs are complete
// before any of its kernels start.
PPD_DEV void pdl_release() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
PPD_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Running log-sum-exp of a row: maximum m, sum s of exp(x - m) over the finite
// entries, and whether a NaN or +inf was seen.  -inf entries add nothing and
// every exponent is a difference <= 0, so nothing overflows.
struct LseAcc {
    float m, s;
    int bad;
};

PPD_DEV void lse_add(LseAcc &a, float x)
{
    if (isnan(x) || x == INFINITY) {
        a.bad = 1;
    } else if (x > a.m) {
        a.s = a.s * exp2f((a.m - x) * kLog2e) + 1.f;
        a.m = x;
    } else if (x > -INFINITY) {
        a.s += exp2f((x - a.m) * kLog2e);
    }
}

PPD_DEV void lse_merge(LseAcc &a, float om, float os, int ob)
{
    const float nm = fmaxf(a.m, om);
    if (nm > -INFINITY)
        a.s = (a.m > -INFINITY ? a.s * exp2f((a.m - nm) * kLog2e) : 0.f) +
              (om > -INFINITY ? os * exp2f((om - nm) * kLog2e) : 0.f);
    a.m = nm;
    a.bad |= ob;
}

// Merge across the lanes of a warp (every lane ends with the total).
PPD_DEV void lse_warp(LseAcc &a)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, a.m, off);
        const float os = __shfl_xor_sync(0xffffffffu, a.s, off);
        const int ob = __shfl_xor_sync(0xffffffffu, a.bad, off);
        lse_merge(a, om, os, ob);
    }
}

// The K-th entry of a best-K list: the one a new entry must beat.
struct TopkEdge {
    float v;
    int i;
};

// Insert (x, v) into a best-K list (best first) that it is known to enter, and
// return the list's new K-th entry.  Out of line: the score loops test each
// candidate against the K-th entry inline and call this rarely (a few dozen
// times per thread), so one copy of the insertion keeps their code within the
// instruction cache.
__device__ __noinline__ TopkEdge topk_insert_slow(float *hv, int *hi, int K, float x, int v)
{
    float cv = x;
    int ci = v;
    for (int r = 0; r < K; ++r) {
        if (ranks_before(cv, ci, hv[r], hi[r])) {
            const float sv = hv[r];
            const int si = hi[r];
            hv[r] = cv;
            hi[r] = ci;
            cv = sv;
            ci = si;
        }
    }
    return TopkEdge{hv[K - 1], hi[K - 1]};
}

PPD_DEV void topk_insert(float *hv, int *hi, TopkEdge &edge, int K, float x, int v)
{
    if (ranks_before(x, v, edge.v, edge.i)) edge = topk_insert_slow(hv, hi, K, x, v);
}

// The best entry over the lanes of a warp (value, index, and the lane holding it).
PPD_DEV void warp_best(float &bv, int &bi, int &bl)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        const int ol = __shfl_xor_sync(0xffffffffu, bl, off);
        if (ranks_before(ov, oi, bv, bi)) {
            bv = ov;
            bi = oi;
            bl = ol;
        }
    }
}

// The n_ept prompt chains below sequence b's accepted end node, for chain
// position d (one block of kTopkThreads threads, T <= kTopkThreads): each
// node's lowest-index prompt child (a later node) by a shared-memory minimum,
// one node per thread; the end node's prompt children ranked by ballots; each
// chain walked through those links.  Leaves in c the chains' nodes at
// position d and the state k (0 with fewer than n_ept heads, else the
// shortest chain capped at n_states - 1); ends with a block barrier.
struct ChainSmem {
    int fc[kMaxTree];
    int head[kNextMaxEpt], len[kNextMaxEpt], node[kNextMaxEpt];
    int wcnt[kTopkWarps];
    int nh, k;
};

PPD_DEV void find_chains(ChainSmem &c, const int32_t *parent, const int32_t *cand,
                         const int32_t *path, const int32_t *accept_len, int b, int d, int T,
                         int n_states, int n_ept)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int cap = n_states - 1;
    const int32_t *par = parent + (size_t)b * T;
    const int32_t *tok = cand + (size_t)b * T;
    const int n = __ldg(accept_len + b);
    const int e = (n >= 1 && n <= T) ? __ldg(path + (size_t)b * T + n - 1) : -1;
    for (int i = tid; i < T; i += kTopkThreads) c.fc[i] = INT_MAX;
    __syncthreads();
    bool head = false;
    if (tid < T) {
        const int pa = __ldg(par + tid), tk = __ldg(tok + tid);
        if (tk == -1 && pa >= 0 && pa < tid) atomicMin(c.fc + pa, tid);
        head = tk == -1 && e >= 0 && e < T && pa == e && tid > e;
    }
    const unsigned hm = __ballot_sync(0xffffffffu, head);
    if (lane == 0) c.wcnt[warp] = __popc(hm);
    __syncthreads();
    int rank = __popc(hm & ((1u << lane) - 1u));
    for (int w = 0; w < warp; ++w) rank += c.wcnt[w];
    if (head && rank < n_ept) c.head[rank] = tid;
    if (tid == 0) {
        int cnt = 0;
        for (int w = 0; w < kTopkWarps; ++w) cnt += c.wcnt[w];
        c.nh = min(cnt, n_ept);
    }
    __syncthreads();
    // each chain's length (capped) and its node at position d, one thread a chain
    if (c.nh == n_ept) {
        for (int j = tid; j < n_ept; j += kTopkThreads) {
            int cur = c.head[j], len = 1, node = d == 1 ? cur : -1;
            while (len < cap) {
                const int nx = c.fc[cur];
                if (nx == INT_MAX) break;
                cur = nx;
                ++len;
                if (len == d) node = cur;
            }
            c.len[j] = len;
            c.node[j] = node;
        }
    }
    __syncthreads();
    if (tid == 0) {
        int k = 0;
        if (c.nh == n_ept) {
            k = cap;
            for (int j = 0; j < n_ept; ++j) k = min(k, c.len[j]);
        }
        c.k = k;
    }
    __syncthreads();
}

// ln sum_v exp(x_j[v]) of chain row j = blockIdx.z at position d of sequence b
// (probability mode): an online maximum and sum per thread, merged over the
// block; NaN when the row holds a NaN or +inf, or only -inf.  Written to
// lse[(b * (n_states - 1) + d - 1) * kNextMaxEpt + j].
__global__ void __launch_bounds__(kTopkThreads)
next_lse_kernel(const float *__restrict__ logits, const int32_t *parent, const int32_t *cand,
                const int32_t *path, const int32_t *accept_len, int T, int V, int n_states,
                int n_ept, int vec, float *lse)
{
    __shared__ ChainSmem cs;
    __shared__ float s_m[kTopkWarps], s_s[kTopkWarps];
    __shared__ int s_b[kTopkWarps];
    const int b = blockIdx.x, d = blockIdx.y + 1, j = blockIdx.z;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    pdl_release();
    find_chains(cs, parent, cand, path, accept_len, b, d, T, n_states, n_ept);
    if (d > cs.k) return;   // uniform over the block
    const float *x = logits + ((size_t)b * T + cs.node[j]) * V;
    LseAcc acc{-INFINITY, 0.f, 0};
    if (vec) {
        const int V4 = V >> 2;
        for (int v4 = tid; v4 < V4; v4 += kBatch * kTopkThreads) {
            float4 xs[kBatch];
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                xs[q] = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
                if (v4 + q * kTopkThreads < V4) xs[q] = __ldg(reinterpret_cast<const float4 *>(x) + v4 + q * kTopkThreads);
            }
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                lse_add(acc, xs[q].x);
                lse_add(acc, xs[q].y);
                lse_add(acc, xs[q].z);
                lse_add(acc, xs[q].w);
            }
        }
    } else {
        for (int v = tid; v < V; v += kTopkThreads) lse_add(acc, __ldg(x + v));
    }
    lse_warp(acc);
    if (lane == 0) {
        s_m[warp] = acc.m;
        s_s[warp] = acc.s;
        s_b[warp] = acc.bad;
    }
    __syncthreads();
    if (warp == 0) {
        LseAcc a{-INFINITY, 0.f, 0};
        if (lane < kTopkWarps) a = LseAcc{s_m[lane], s_s[lane], s_b[lane]};
        lse_warp(a);
        if (lane == 0)
            lse[((size_t)b * (n_states - 1) + d - 1) * kNextMaxEpt + j] =
                (a.bad || a.m == -INFINITY) ? NAN : a.m + logf(a.s);
    }
}

// Top-K (K <= kNextMaxK) of the averaged logits (ept_mean 0) or probabilities
// (ept_mean 1) over columns [z * chunk, (z + 1) * chunk) at chain position d
// (1-based) of sequence b, z = blockIdx.z, written to the partial lists
// part_*[((b * (n_states - 1) + d - 1) * gridDim.z + z) * K ...] in ranking
// order (NaN first, then larger value, then lower index).  The first block of
// position 1 also writes the state k of its sequence to kstate[b].  vec: rows
// may be read as float4 (chunk is then a multiple of 4).
__global__ void __launch_bounds__(kTopkThreads)
next_topk_kernel(const float *__restrict__ logits, const int32_t *parent, const int32_t *cand,
                 const int32_t *path, const int32_t *accept_len, int T, int V, int n_states, int K,
                 int n_ept, int ept_mean, int vec, int chunk, const float *lse, float *part_val,
                 int32_t *part_idx, int32_t *kstate)
{
    __shared__ ChainSmem cs;
    __shared__ float s_lse[kNextMaxEpt];
    __shared__ float s_lv[kTopkWarps][kNextMaxK];
    __shared__ int s_li[kTopkWarps][kNextMaxK];
    const int b = blockIdx.x;
    const int d = blockIdx.y + 1;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    pdl_release();
    find_chains(cs, parent, cand, path, accept_len, b, d, T, n_states, n_ept);
    pdl_wait();   // the log-sum-exps, and the previous call's readers of kstate and the lists
    if (tid == 0 && d == 1 && blockIdx.z == 0) kstate[b] = cs.k;
    if (d > cs.k) return;   // uniform over the block
    auto row = [&](int j) { return logits + ((size_t)b * T + cs.node[j]) * V; };
    const bool probs = ept_mean == 1 && n_ept > 1;
    const int c0 = (int)blockIdx.z * chunk, c1 = min(V, c0 + chunk);   // this block's columns

    // ---- probability mode: the chain rows' log-sum-exps (next_lse_kernel)
    if (probs) {
        for (int j = tid; j < n_ept; j += kTopkThreads)
            s_lse[j] = __ldcg(lse + ((size_t)b * (n_states - 1) + d - 1) * kNextMaxEpt + j);
        __syncthreads();
    }

    // ---- this thread's best K over its columns, best first
    float hv[kNextMaxK];
    int hi[kNextMaxK];
#pragma unroll
    for (int r = 0; r < kNextMaxK; ++r) {
        hv[r] = -INFINITY;
        hi[r] = INT_MAX;
    }
    TopkEdge edge{-INFINITY, INT_MAX};
    const float n_f = (float)n_ept;
    if (vec) {
        const int e4 = c1 >> 2;
        for (int base = (c0 >> 2) + tid; base < e4; base += kBatch * kTopkThreads) {
            float4 sc[kBatch];
#pragma unroll
            for (int q = 0; q < kBatch; ++q) sc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (probs) {
                // sum_j p_j(v), chain order; a NaN lse_j makes every score NaN
                for (int j = 0; j < n_ept; ++j) {
                    const float4 *x4 = reinterpret_cast<const float4 *>(row(j));
                    const float l = s_lse[j];
                    float4 x[kBatch];
#pragma unroll
                    for (int q = 0; q < kBatch; ++q) x[q] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int q = 0; q < kBatch; ++q)
                        if (base + q * kTopkThreads < e4) x[q] = __ldcs(x4 + base + q * kTopkThreads);
#pragma unroll
                    for (int q = 0; q < kBatch; ++q) {
                        if (base + q * kTopkThreads < e4) {
                            sc[q].x += exp2f((x[q].x - l) * kLog2e);
                            sc[q].y += exp2f((x[q].y - l) * kLog2e);
                            sc[q].z += exp2f((x[q].z - l) * kLog2e);
                            sc[q].w += exp2f((x[q].w - l) * kLog2e);
                        }
                    }
                }
            } else {
                // the EPT average: summed in chain order, then one IEEE division
                const float4 *x0 = reinterpret_cast<const float4 *>(row(0));
#pragma unroll
                for (int q = 0; q < kBatch; ++q)
                    if (base + q * kTopkThreads < e4) sc[q] = __ldcs(x0 + base + q * kTopkThreads);
                if (n_ept > 1) {
                    for (int j = 1; j < n_ept; ++j) {
                        const float4 *x4 = reinterpret_cast<const float4 *>(row(j));
                        float4 x[kBatch];
#pragma unroll
                        for (int q = 0; q < kBatch; ++q) {
                            x[q] = make_float4(0.f, 0.f, 0.f, 0.f);
                            if (base + q * kTopkThreads < e4) x[q] = __ldcs(x4 + base + q * kTopkThreads);
                        }
#pragma unroll
                        for (int q = 0; q < kBatch; ++q) {
                            sc[q].x += x[q].x;
                            sc[q].y += x[q].y;
                            sc[q].z += x[q].z;
                            sc[q].w += x[q].w;
                        }
                    }
#pragma unroll
                    for (int q = 0; q < kBatch; ++q) {
                        sc[q].x = sc[q].x / n_f;
                        sc[q].y = sc[q].y / n_f;
                        sc[q].z = sc[q].z / n_f;
                        sc[q].w = sc[q].w / n_f;
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < kBatch; ++q) {
                const int v4 = base + q * kTopkThreads;
                if (v4 < e4) {
                    topk_insert(hv, hi, edge, K, sc[q].x, 4 * v4);
                    topk_insert(hv, hi, edge, K, sc[q].y, 4 * v4 + 1);
                    topk_insert(hv, hi, edge, K, sc[q].z, 4 * v4 + 2);
                    topk_insert(hv, hi, edge, K, sc[q].w, 4 * v4 + 3);
                }
            }
        }
    } else {
        for (int v = c0 + tid; v < c1; v += kTopkThreads) {
            float xv;
            if (probs) {
                xv = 0.f;
                for (int j = 0; j < n_ept; ++j) xv += exp2f((__ldcs(row(j) + v) - s_lse[j]) * kLog2e);
            } else {
                xv = __ldcs(row(0) + v);
                if (n_ept > 1) {
                    for (int j = 1; j < n_ept; ++j) xv += __ldcs(row(j) + v);
                    xv = xv / n_f;
                }
            }
            topk_insert(hv, hi, edge, K, xv, v);
        }
    }

    // ---- each warp's best K (K rounds: the best head over the lanes, its lane
    // pops it), then warp 0 takes the best K of the warps' lists
    for (int r = 0; r < K; ++r) {
        float bv = hv[0];
        int bi = hi[0], bl = lane;
        warp_best(bv, bi, bl);
        if (lane == 0) {
            s_lv[warp][r] = bv;
            s_li[warp][r] = bi;
        }
        if (lane == bl) {
            for (int q = 0; q + 1 < K; ++q) {
                hv[q] = hv[q + 1];
                hi[q] = hi[q + 1];
            }
            hv[K - 1] = -INFINITY;
            hi[K - 1] = INT_MAX;
        }
    }
    __syncthreads();
    if (warp == 0) {
        int ptr = 0;   // lane w: next entry of warp w's list
        for (int r = 0; r < K; ++r) {
            float bv = -INFINITY;
            int bi = INT_MAX, bl = lane;
            if (lane < kTopkWarps && ptr < K) {
                bv = s_lv[lane][ptr];
                bi = s_li[lane][ptr];
            }
            warp_best(bv, bi, bl);
            if (lane == 0) {
                const size_t o = (((size_t)b * (n_states - 1) + d - 1) * gridDim.z + blockIdx.z) * K + r;
                part_val[o] = bv;
                part_idx[o] = bi;
            }
            if (lane == bl) ++ptr;
        }
    }
}

// One warp per (sequence b, chain position d <= its state): the best K of the
// n_split partial lists, in ranking order, into topk[(b * (n_states - 1) + d -
// 1) * K ...].  Lane z walks list z.
__global__ void __launch_bounds__(32)
next_topk_merge_kernel(const float *part_val, const int32_t *part_idx, int n_states, int K,
                       int n_split, const int32_t *kstate, int32_t *topk)
{
    const int b = blockIdx.x, d = blockIdx.y + 1, lane = threadIdx.x;
    pdl_release();
    pdl_wait();   // the partial lists and the states
    if (d > __ldcg(kstate + b)) return;   // uniform over the warp
    const size_t base = ((size_t)b * (n_states - 1) + d - 1) * n_split;
    int ptr = 0;
    for (int r = 0; r < K; ++r) {
        float bv = -INFINITY;
        int bi = INT_MAX, bl = lane;
        if (lane < n_split && ptr < K) {
            bv = __ldcg(part_val + (base + lane) * K + ptr);
            bi = __ldcg(part_idx + (base + lane) * K + ptr);
        }
        warp_best(bv, bi, bl);
        if (lane == 0) topk[((size_t)b * (n_states - 1) + d - 1) * K + r] = bi;
        if (lane == bl) ++ptr;
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
    pdl_wait();   // the states and the guesses
    int k = 0;
    if (!bad) {
        const int e = __ldg(path + (size_t)b * T + n - 1);
        bad = !(e >= 0 && e < T);
        if (!bad && n_states > 1) k = __ldcg(kstate + b);
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
                    tokv = __ldcg(topk + ((size_t)b * (n_states - 1) + depth - 1) * K + r);
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

// A kernel launch, as a programmatic dependent of the stream's previous grid
// when `chained` (it may then start before that grid completes, and waits
// for it with griddepcontrol.wait).
template <typename... KArgs, typename... Args>
static cudaError_t launch_chained(void (*kern)(KArgs...), dim3 grid, dim3 block, bool chained,
                                  cudaStream_t stream, Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = chained ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

cudaError_t launch_next_tree(const float *logits, const int32_t *parent, const int32_t *cand,
                             const int32_t *path, const int32_t *accept_len,
                             const int32_t *next_token, int B, int T, int V, int n_states,
                             int T_next, const int32_t *tmpl_parent, const int32_t *tmpl_rank, int K,
                             int n_ept, int ept_mean, int32_t *topk, int32_t *kstate,
                             float *part_val, int32_t *part_idx, float *lse, int num_sms,
                             int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                             int32_t *status, cudaStream_t stream)
{
    bool chained = false;   // the call's first kernel waits for the work before it
    if (n_states > 1) {
        const int vec = (V % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
        // each row shared by n_split blocks, about two blocks per SM in all
        const long long rows = (long long)B * (n_states - 1);
        int n_split = (int)((2LL * num_sms + rows - 1) / rows);
        n_split = n_split < 1 ? 1 : (n_split > kNextMaxSplit ? kNextMaxSplit : n_split);
        int chunk = (V + n_split - 1) / n_split;
        chunk = (chunk + 3) & ~3;
        n_split = (V + chunk - 1) / chunk;
        const unsigned cap = (unsigned)(n_states - 1);
        cudaError_t e;
        if (ept_mean == 1 && n_ept > 1) {
            e = launch_chained(next_lse_kernel, dim3((unsigned)B, cap, (unsigned)n_ept),
                               dim3(kTopkThreads), chained, stream, logits, parent, cand, path,
                               accept_len, T, V, n_states, n_ept, vec, lse);
            if (e != cudaSuccess) return e;
            chained = true;
        }
        e = launch_chained(next_topk_kernel, dim3((unsigned)B, cap, (unsigned)n_split),
                           dim3(kTopkThreads), chained, stream, logits, parent, cand, path,
                           accept_len, T, V, n_states, K, n_ept, ept_mean, vec, chunk,
                           (const float *)lse, part_val, part_idx, kstate);
        if (e != cudaSuccess) return e;
        e = launch_chained(next_topk_merge_kernel, dim3((unsigned)B, cap), dim3(32), true, stream,
                           (const float *)part_val, (const int32_t *)part_idx, n_states, K, n_split,
                           (const int32_t *)kstate, topk);
        if (e != cudaSuccess) return e;
        chained = true;
    }
    return launch_chained(next_assemble_kernel, dim3((unsigned)((B + 3) / 4)), dim3(128), chained,
                          stream, parent, cand, path, accept_len, next_token, B, T, n_states,
                          T_next, tmpl_parent, tmpl_rank, K, (const int32_t *)topk,
                          (const int32_t *)kstate, next_parent, next_cand, next_state, status);
}

}  // namespace ppd
