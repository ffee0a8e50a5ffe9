// ppd_attention_common.cuh -- pieces shared by the two tree-attention kernels
// (ppd_attention.cu for trees of up to 64 tokens, ppd_attention_rows.cu for
// 65..512): the work split and unit walk, drain waits, mask kinds and the
// fused step's side warp.
#pragma once

#include "ppd_accept.cuh"
#include "ppd_device.cuh"
#include "ppd_kernels.h"

#include <algorithm>
#include <atomic>
#include <type_traits>

namespace ppd {

// A (layer, sequence, head) unit: its sequence, clamped prefix length and tiles
// (prefix tiles of 128 keys, then one tile of the tree's own keys).
struct UnitInfo {
    int lbh, qb, b, P, P_raw, n_pref, n_tiles;
};

// Unit u = (layer, sequence, head) slice lbh and block qb of its query rows
// (slices of trees over 128 tokens split their queries into blocks of 128).
PPD_DEV UnitInfo unit_info(const AttnParams &p, int u)
{
    UnitInfo ui;
    ui.lbh = u / p.n_qb;
    ui.qb = u - ui.lbh * p.n_qb;
    ui.b = (ui.lbh / p.H) % p.B;
    ui.P_raw = __ldg(p.prefix_len + ui.b);
    ui.P = min(max(ui.P_raw, 0), p.S_max);
    ui.n_pref = (ui.P + 127) >> 7;
    ui.n_tiles = ui.n_pref + p.n_tt;
    return ui;
}

// ------------------------------------------------------------------ work split
//
// Without p.split, units are taken round-robin (CTA c: units c, c+G, c+2G,
// ...), whole.  With p.split (launches with fewer units than CTAs, where whole
// units would leave SMs idle) all units are shared out by their key tiles: the
// tiles (unit u's tiles 0..n_tiles(u)-1, units in order) go to the CTAs in
// equal contiguous ranges (CTA c: tiles [c*N/G, (c+1)*N/G)).  A unit cut by a
// range boundary is done in parts, one per CTA; each part leaves its partial
// softmax state (the unnormalised O rows, the running maximum and the row sum
// of every query) in a slot of its CTA, and the CTA holding the unit's first
// tile leaves a record of it.  Once the launch is complete a second, small
// grid merges every recorded unit, so nothing in the attention grid waits
// for, or counts, other CTAs.

struct WorkRange {
    int rr_units;            // units taken whole, round-robin (all, or none)
    int u_first, j_first;    // first unit and tile of this CTA's range (split)
    int n_tiles;             // tiles in the range (0: none)
    int u_last;              // last unit the range touches
    long long x_first;       // index of the range's first tile
    long long n_tail;        // tiles shared out by the split
};

// First tail tile of CTA c, and the CTA holding tail tile x.
PPD_DEV long long split_start(int c, long long N, int G) { return (long long)c * N / G; }
PPD_DEV int split_cta_of(long long x, long long N, int G) { return (int)(((x + 1) * G + N - 1) / N) - 1; }

// This CTA's work, computed by one whole warp (every lane gets the result).
// The tiles of one layer's block of sequence b number H * n_qb * (n_pref(b) +
// n_tt); lanes hold sequences b = lane and lane + 32.  kHint: the prefix
// lengths are read through L2 because they may still be changing (a plan
// made before the wait of a chained launch, used for prefetch hints only).
template <bool kHint = false>
PPD_DEV WorkRange plan_range(const AttnParams &p, int lane)
{
    WorkRange w{};
    const int G = (int)gridDim.x, c = (int)blockIdx.x;
    // no tail range unless one is found below
    w.u_first = p.n_units;
    w.u_last = -1;
    w.n_tiles = 0;
    w.rr_units = p.split ? 0 : p.n_units;   // units taken whole, round-robin
    if (!p.split) return w;
    const unsigned full = 0xffffffffu;
    const int per_b = p.H * p.n_qb;
    auto nt_of = [&](int b) {
        const int P = min(max(kHint ? ld_relaxed_gpu_s32(p.prefix_len + b) : __ldg(p.prefix_len + b), 0),
                          p.S_max);
        return ((P + 127) >> 7) + p.n_tt;
    };
    const int w0 = lane < p.B ? per_b * nt_of(lane) : 0;
    const int w1 = lane + 32 < p.B ? per_b * nt_of(lane + 32) : 0;
    int s0 = w0, s1 = w1;   // inclusive prefix sums over b
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int a = __shfl_up_sync(full, s0, o);
        const int x = __shfl_up_sync(full, s1, o);
        if (lane >= o) {
            s0 += a;
            s1 += x;
        }
    }
    s1 += __shfl_sync(full, s0, 31);
    const long long per_layer = __shfl_sync(full, s1, 31);
    const long long N = per_layer * p.L;
    // global tile index of unit u's tile 0
    auto origin = [&](int u) {
        const int l = u / (p.B * per_b);
        const int rem = u - l * p.B * per_b;
        const int b = rem / per_b, idx = rem - b * per_b;
        const int incl = b < 32 ? __shfl_sync(full, s0, b & 31) : __shfl_sync(full, s1, b & 31);
        const int wt = b < 32 ? __shfl_sync(full, w0, b & 31) : __shfl_sync(full, w1, b & 31);
        return (long long)l * per_layer + (incl - wt) + (long long)idx * (wt / per_b);
    };
    // unit and tile of global tile x (0 <= x < N)
    auto locate = [&](long long x, int &u, int &j) {
        const int l = (int)(x / per_layer);
        const int r = (int)(x - (long long)l * per_layer);
        const unsigned m0 = __ballot_sync(full, lane < p.B && s0 > r);
        int b, incl, wt;
        if (m0) {
            b = __ffs(m0) - 1;
            incl = __shfl_sync(full, s0, b);
            wt = __shfl_sync(full, w0, b);
        } else {
            const unsigned m1 = __ballot_sync(full, lane + 32 < p.B && s1 > r);
            const int bl = m1 ? __ffs(m1) - 1 : 0;
            b = bl + 32;
            incl = __shfl_sync(full, s1, bl);
            wt = __shfl_sync(full, w1, bl);
        }
        const int rb = r - (incl - wt);   // tile offset within the block of sequence b
        const int nt = wt / per_b;
        const int idx = rb / nt;
        j = rb - idx * nt;
        u = (l * p.B + b) * per_b + idx;
    };
    const long long base = origin(w.rr_units);
    w.n_tail = N - base;
    const long long gs = split_start(c, w.n_tail, G), ge = split_start(c + 1, w.n_tail, G);
    w.x_first = gs;
    w.n_tiles = (int)(ge - gs);
    if (ge > gs) {
        int jl;
        locate(base + gs, w.u_first, w.j_first);
        locate(base + ge - 1, w.u_last, jl);
    }
    return w;
}

// Before the wait of a chained launch (one warp, all lanes): ask L2 for the
// first `n` K and V prefix tiles this CTA will stream, from a plan made with
// prefix lengths that may still be changing.  Only a hint -- nothing is
// written to shared memory and nothing waits on it; the real loads follow the
// wait with the plan remade -- so the preceding grid's work overlaps the
// first tiles' trip from HBM.  Tree tiles are skipped (in a model the
// preceding grids write them).
template <bool SPLIT>
PPD_DEV void prefetch_first_tiles(const AttnParams &p, int lane, const CUtensorMap *kc,
                                  const CUtensorMap *vc, int dch, int n)
{
    const WorkRange w = plan_range<true>(p, lane);
    if (lane != 0) return;
    int u = SPLIT ? w.u_first : (int)blockIdx.x;
    int j = SPLIT ? w.j_first : 0;
    int left = SPLIT ? w.n_tiles : n;
    for (int k = 0; k < n && left > 0 && u < p.n_units; ++k, --left) {
        const int lbh = u / p.n_qb;
        const int b = (lbh / p.H) % p.B;
        const int P = min(max(ld_relaxed_gpu_s32(p.prefix_len + b), 0), p.S_max);
        const int n_pref = (P + 127) >> 7;
        if (j < n_pref) {
            for (int c = 0; c < dch; ++c) {
                tma_prefetch_l2_3d(kc, c * 64, j * 128, lbh);
                tma_prefetch_l2_3d(vc, c * 64, j * 128, lbh);
            }
            ++j;
        } else {   // the unit's tree tiles: on to the next unit
            u = SPLIT ? u + 1 : u + (int)gridDim.x;
            j = 0;
        }
    }
}

// One stretch of a unit's tiles [j0, j1) processed by this CTA.
struct Seg {
    UnitInfo ui;
    int u, j0, j1;
};

// Walks this CTA's segments in order (every role of the CTA walks the same
// sequence): whole units round-robin, or (SPLIT) its range of tiles, `left`
// counting the range's tiles not yet handed out.
template <bool SPLIT>
struct SegIter {
    int u, j0, left;
    PPD_DEV explicit SegIter(const WorkRange &w)
    {
        u = SPLIT ? w.u_first : (int)blockIdx.x;
        j0 = SPLIT ? w.j_first : 0;
        left = SPLIT ? w.n_tiles : 0;
    }
    PPD_DEV bool next(const AttnParams &p, Seg &s)
    {
        if (!SPLIT) {
            if (u >= p.n_units) return false;
            s.ui = unit_info(p, u);
            s.u = u;
            s.j0 = 0;
            s.j1 = s.ui.n_tiles;
            u += (int)gridDim.x;
            return true;
        }
        if (left <= 0 || u >= p.n_units) return false;
        s.ui = unit_info(p, u);
        s.u = u;
        s.j0 = j0;
        s.j1 = min(s.ui.n_tiles, j0 + left);
        if (s.j1 <= j0) {   // cannot happen with a consistent plan; never loop on it
            left = 0;
            return false;
        }
        left -= s.j1 - j0;
        ++u;
        j0 = 0;
        return true;
    }
};

// Does the CTA process all of the segment's unit?
PPD_DEV bool seg_whole(const Seg &s) { return s.j0 == 0 && s.j1 == s.ui.n_tiles; }

// Tail-relative index of the segment's unit's tile 0, given the iterator
// right after it handed the (tail) segment out.
template <bool SPLIT>
PPD_DEV long long seg_unit_origin(const WorkRange &w, const SegIter<SPLIT> &it, const Seg &s)
{
    return w.x_first + (w.n_tiles - it.left) - s.j1;
}

// The parts of a cut unit: the CTAs c_a..c_b whose ranges are not empty (a
// launch with fewer tiles than CTAs leaves some ranges empty).  Part c's slot
// is 2c for the first segment of its range and 2c + 1 for the last (only c_a
// can hold the unit in its last segment).
struct SplitParts {
    int c_a, c_b, slot_a, n_parts;
};

PPD_DEV bool split_nonempty(int c, long long N, int G) { return split_start(c + 1, N, G) > split_start(c, N, G); }

PPD_DEV SplitParts split_parts(long long N, long long off, int n_tiles)
{
    SplitParts sp;
    const int G = (int)gridDim.x;
    sp.c_a = split_cta_of(off, N, G);
    sp.c_b = split_cta_of(off + n_tiles - 1, N, G);
    sp.slot_a = 2 * sp.c_a + (split_start(sp.c_a, N, G) < off ? 1 : 0);
    sp.n_parts = 0;
    for (int c = sp.c_a; c <= sp.c_b; ++c) sp.n_parts += split_nonempty(c, N, G) ? 1 : 0;
    return sp;
}

PPD_DEV int split_slot(const SplitParts &sp, int c) { return c == sp.c_a ? sp.slot_a : 2 * c; }

// Floats of one partial-state slot: kSplitRows rows of D, their maxima, their sums.
PPD_DEV size_t split_slot_floats(int D) { return (size_t)kSplitRows * (D + 2); }

// Merge the partial states of a cut unit whose parts have all arrived: slot
// row r (output row out_row0 + r), columns [c0, c0 + 8), by one thread.  One
// pass over the parts with a running maximum M: part c enters with weight
// 2^(m_c - M), earlier sums are rescaled when M grows; the output is the
// weighted sum of the parts' O rows over the weighted sum of their row sums.
// The parts are read eight at a time, every load of a batch issued before any
// is used, so a batch costs one round trip to L2.
static __device__ __forceinline__ void split_merge_chunk(const float *split_part, float *out, float *lse,
                                                         const SplitParts &sp, long long N, int G,
                                                         size_t out_row0, int r, int c0, int D)
{
    constexpr int PB = 8;   // parts per batch
    const size_t sf = split_slot_floats(D);
    const bool dense = N >= G;   // no empty ranges
    float M = -INFINITY, Ls = 0.f;
    float acc[8];
#pragma unroll
    for (int x = 0; x < 8; ++x) acc[x] = 0.f;
    for (int cb = sp.c_a; cb <= sp.c_b; cb += PB) {
        float mc[PB], lc[PB];
        float4 v[PB][2];
#pragma unroll
        for (int y = 0; y < PB; ++y) {
            const int c = cb + y;
            const bool live = c <= sp.c_b && (dense || split_nonempty(c, N, G));
            const float *b_ = split_part + (size_t)split_slot(sp, live ? c : sp.c_a) * sf;
            mc[y] = live ? __ldcg(b_ + (size_t)kSplitRows * D + r) : -INFINITY;
            lc[y] = live ? __ldcg(b_ + (size_t)kSplitRows * D + kSplitRows + r) : 0.f;
            const float4 *o4 = reinterpret_cast<const float4 *>(b_ + (size_t)r * D + c0);
            v[y][0] = live ? __ldcg(o4) : make_float4(0.f, 0.f, 0.f, 0.f);
            v[y][1] = live ? __ldcg(o4 + 1) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int y = 0; y < PB; ++y) {
            if (mc[y] == -INFINITY) continue;   // absent, or the part saw no key of this row
            const float Mn = fmaxf(M, mc[y]);
            const float so = ex2(M - Mn);       // 0 while M = -inf
            const float w = ex2(mc[y] - Mn);
            Ls = fmaf(Ls, so, w * lc[y]);
#pragma unroll
            for (int x = 0; x < 2; ++x) {
                acc[4 * x] = fmaf(acc[4 * x], so, w * v[y][x].x);
                acc[4 * x + 1] = fmaf(acc[4 * x + 1], so, w * v[y][x].y);
                acc[4 * x + 2] = fmaf(acc[4 * x + 2], so, w * v[y][x].z);
                acc[4 * x + 3] = fmaf(acc[4 * x + 3], so, w * v[y][x].w);
            }
            M = Mn;
        }
    }
    const float inv = 1.f / Ls;
    float *dst = out + (out_row0 + r) * D + c0;
    if ((reinterpret_cast<uintptr_t>(out) & 15u) == 0) {
        reinterpret_cast<float4 *>(dst)[0] = make_float4(acc[0] * inv, acc[1] * inv, acc[2] * inv, acc[3] * inv);
        reinterpret_cast<float4 *>(dst)[1] = make_float4(acc[4] * inv, acc[5] * inv, acc[6] * inv, acc[7] * inv);
    } else {
#pragma unroll
        for (int x = 0; x < 8; ++x) dst[x] = acc[x] * inv;
    }
    if (c0 == 0 && lse) lse[out_row0 + r] = (M + lg2(Ls)) * 0.69314718055994530942f;
}

PPD_DEV void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
                 "r"(d)
                 : "memory");
}

// Time-bounded wait that ignores the abort flag (used only to drain copies
// still in flight after an abort, before the CTA exits).
PPD_DEV void mbar_wait_drain(uint64_t *bar, uint32_t parity)
{
    const uint32_t a = smem_addr(bar);
    const uint64_t t0 = global_timer();
    while (!mbar_try_wait(a, parity))
        if (global_timer() - t0 > kWaitLimitNs) return;
}

template <int K>
using kind_t = std::integral_constant<int, K>;

// Mask kinds of a tile: every key visible (a full prefix tile), keys t < n_valid
// visible (the last, partial prefix tile), or the tree-ancestor mask.
enum : int { kMaskNone = 0, kMaskRows = 1, kMaskTree = 2 };

// One warp's partial top-1 of columns [lo, hi) of the logits row x, and with
// kStats the softmax statistics of the same columns at scale stat_k; lane 0
// holds the result.  Four 16-byte loads per lane (2 KB per warp) are in
// flight at a time: deeper bursts of loads from this warp slow the softmax
// warps that share its SM sub-partition more than they gain.
template <bool kStats>
PPD_DEV void warp_logit_partial(const float *x, int lo, int hi, bool vec, float stat_k, int lane,
                                float &bv, int &bi, SoftStats &st)
{
    bv = -INFINITY;
    bi = INT_MAX;
    st = SoftStats{};
    auto take4 = [&](const float4 &f, int base) {
        consider(f.x, base, bv, bi);
        consider(f.y, base + 1, bv, bi);
        consider(f.z, base + 2, bv, bi);
        consider(f.w, base + 3, bv, bi);
        if (kStats) stats_add4(st, f.x * stat_k, f.y * stat_k, f.z * stat_k, f.w * stat_k);
    };
    if (vec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(x);
        const int n4_hi = hi >> 2;
        int i = (lo >> 2) + lane;
        for (; i + 3 * 32 < n4_hi; i += 4 * 32) {
            float4 f[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) f[k] = __ldcs(x4 + i + k * 32);
#pragma unroll
            for (int k = 0; k < 4; ++k) take4(f[k], 4 * (i + k * 32));
        }
        for (; i < n4_hi; i += 32) take4(__ldcs(x4 + i), 4 * i);
    } else {
        for (int i = lo + lane; i < hi; i += 32) {
            const float v = __ldcs(x + i);
            consider(v, i, bv, bi);
            if (kStats) stats_add4(st, v * stat_k, -INFINITY, -INFINITY, -INFINITY);
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

// In-grid argmax of the fused step: this CTA's chunks of the [B*T][splits]
// partial grid (chunk c by CTA c mod grid), then its flag.  Each lane fences
// its own writes before the warp barrier, so lane 0's release covers them all.
PPD_DEV void side_argmax_chunks(const AttnParams &p, unsigned long long tag, int lane)
{
    const FusedStep &f = p.fs;
    const int S = f.splits;
    const long long n_chunks = (long long)p.B * p.T * S;
    for (long long c = blockIdx.x; c < n_chunks; c += gridDim.x) {
        const long long row = c / S;
        const int lo = (int)(c - row * S) * f.chunk;
        const int hi = min(f.V, lo + f.chunk);
        const float *x = f.logits + row * (long long)f.V;
        float bv;
        int bi;
        SoftStats st;
        if (f.typical) warp_logit_partial<true>(x, lo, hi, f.vec != 0, f.stat_k, lane, bv, bi, st);
        else warp_logit_partial<false>(x, lo, hi, f.vec != 0, 0.f, lane, bv, bi, st);
        if (lane == 0) {
            f.part_val[c] = bv;
            f.part_idx[c] = bi;
            if (f.typical) {
                float *ps = f.part_stats + 3 * c;
                ps[0] = st.m;
                ps[1] = st.s;
                ps[2] = st.t;
            }
        }
    }
    __threadfence();
    __syncwarp();
    if (lane == 0 && (int)blockIdx.x != f.withhold_cta) st_release_gpu(f.ready + blockIdx.x, tag);
}

// Wait until every CTA of the grid has published `tag` (bounded: raises the
// CTA's abort flag and returns false after f.wait_limit_ns, or at once when the
// flag is already up; lane 0 takes that decision for the whole warp, so no
// lane leaves while others still shuffle).  Only CTA 0 reads the per-CTA flags; once all are up
// it advances the epoch for the next call and publishes `tag` in all_ready,
// the one word the other CTAs poll (from one lane, with a backoff), so the
// waits add little to the L2 traffic of the attention stream.
PPD_DEV bool side_wait_all(const AttnParams &p, unsigned long long tag, int lane,
                           volatile int *abort_flag)
{
    const FusedStep &f = p.fs;
    const int G = (int)gridDim.x;
    const uint64_t t0 = global_timer();
    bool done = false;
    while (true) {
        if (blockIdx.x == 0) {
            bool ok = true;
            for (int c = lane; c < G; c += 32) ok = ok && ld_acquire_gpu(f.ready + c) == tag;
            done = __all_sync(0xffffffffu, ok);
        } else {
            done = __shfl_sync(0xffffffffu, lane == 0 && ld_acquire_gpu(f.all_ready) == tag, 0);
        }
        if (done) break;
        const bool give_up = __shfl_sync(
            0xffffffffu, lane == 0 && (*abort_flag || global_timer() - t0 > f.wait_limit_ns), 0);
        if (give_up) {
            if (lane == 0) *abort_flag = 1;
            return false;
        }
        __nanosleep(blockIdx.x == 0 ? 200 : 1000);
    }
    __syncwarp();
    __threadfence();
    if (blockIdx.x == 0 && lane == 0) {
        st_relaxed_gpu(f.epoch, tag);
        st_release_gpu(f.all_ready, tag);
    }
    return true;
}

// Side work of the fused verification step, done by one extra warp of every CTA
// while the other warps stream attention.  Once the argmax partials are
// complete -- the preceding grid's (griddepcontrol.wait), or with in_grid the
// ones the side warps of all CTAs compute first (side_argmax_chunks, then
// side_wait_all) -- for every sequence b this CTA touches, or is designated to
// report (b mod grid), the warp combines the node argmax from the partial
// maxima, decides acceptance, writes the sequence's outputs if designated, and
// copies the accepted tree K/V rows of this CTA's own (layer, sequence, head)
// slices into the cache.  Attention only reads cache rows below each prefix,
// so the copies never race with it.  Scratch (parent copies, top-1 tokens,
// path) lives in a per-CTA slice of the workspace.  Kept out of line so that
// its code does not reshape the register allocation of the attention loops.
template <bool kSmallTree>
static __device__ __noinline__ void fused_side_warp(const AttnParams &p, const WorkRange &wr, int lane,
                                                    volatile int *abort_flag)
{
    const FusedStep &f = p.fs;
    unsigned long long tag = 0;
    bool have_all = false;
    if (f.in_grid) {
        tag = __shfl_sync(0xffffffffu, lane == 0 ? ld_relaxed_gpu(f.epoch) + 1ull : 0ull, 0);
        side_argmax_chunks(p, tag, lane);
    } else {
        asm volatile("griddepcontrol.wait;" ::: "memory");
        have_all = true;
    }
    // the units whose first tile this CTA streams (its round-robin units and the
    // tail units starting in its range) compact their slices here
    const int t_lo = wr.u_first + (wr.j_first > 0 ? 1 : 0), t_hi = wr.n_tiles > 0 ? wr.u_last : -1;
    auto owns_first_tile = [&](auto fn) {
        for (int u = (int)blockIdx.x; u < wr.rr_units; u += (int)gridDim.x)
            if (fn(u)) return;
        for (int u = t_lo; u <= t_hi; ++u)
            if (fn(u)) return;
    };
    const int T = p.T, B = p.B, S = f.splits;
    int *s_par = f.scratch + (size_t)blockIdx.x * kSideScratchInts;
    int *top = s_par + kAcceptScratchInts;
    int *path = top + kMaxTree;
    float *s_lse = reinterpret_cast<float *>(path + kMaxTree);
    float *s_ent = s_lse + kMaxTree;
    const int chunks = f.row_bytes >> 4;
    for (int b = 0; b < B; ++b) {
        const bool designated = (b % (int)gridDim.x) == (int)blockIdx.x;
        bool has_unit = false;
        owns_first_tile([&](int u) {
            has_unit = ((u / p.n_qb / p.H) % B) == b && u % p.n_qb == 0;
            return has_unit;
        });
        if (!designated && !has_unit) continue;
        if (!have_all) {
            if (!side_wait_all(p, tag, lane, abort_flag)) return;
            have_all = true;
        }
        // node r's top-1 token from its partials (with typical acceptance also its
        // log-sum-exp and entropy)
        auto row_top = [&](int r, float &lse_r, float &ent_r) {
            const size_t base = ((size_t)b * T + r) * S;
            float bv = -INFINITY;
            int bi = INT_MAX;
            if ((S & 3) == 0) {
                // 16-byte loads, up to 16 partials in flight (the arrays are 256-byte
                // aligned and a row's partials start at a multiple of 4)
                const float4 *v4 = reinterpret_cast<const float4 *>(f.part_val + base);
                const int4 *i4 = reinterpret_cast<const int4 *>(f.part_idx + base);
                for (int k0 = 0; k0 < S / 4; k0 += 4) {
                    float4 v[4];
                    int4 ix[4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if (k0 + j < S / 4) {
                            v[j] = __ldcg(v4 + k0 + j);
                            ix[j] = __ldcg(i4 + k0 + j);
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if (k0 + j < S / 4) {
                            consider(v[j].x, ix[j].x, bv, bi);
                            consider(v[j].y, ix[j].y, bv, bi);
                            consider(v[j].z, ix[j].z, bv, bi);
                            consider(v[j].w, ix[j].w, bv, bi);
                        }
                    }
                }
            } else {
#pragma unroll 8
                for (int k = 0; k < S; ++k) consider(__ldcg(f.part_val + base + k), __ldcg(f.part_idx + base + k), bv, bi);
            }
            if (f.typical) stats_finish(combine_stats(f.part_stats, (int64_t)b * T + r, S), lse_r, ent_r);
            return bi;
        };
        const int32_t *par_b = p.parent + (size_t)b * T;
        const int32_t *tok_b = f.cand_tokens + (size_t)b * T;
        const int P = __ldg(p.prefix_len + b);
        AcceptResult res;
        // the accepted path: in registers (lane j % 32, slot j / 32) for trees of up
        // to 64 nodes, else in the scratch
        int path_r[2] = {-1, -1};
        constexpr bool small = kSmallTree;   // the key-row kernel's trees: T <= 64
        if constexpr (small) {
            int top_r[2] = {0, 0};
            float lse_r[2] = {0.f, 0.f}, ent_r[2] = {0.f, 0.f};
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const int r = lane + 32 * k;
                if (r < T) {
                    top_r[k] = row_top(r, lse_r[k], ent_r[k]);
                    if (designated) f.argmax_out[(size_t)b * T + r] = top_r[k];
                }
            }
            if (f.typical) {
                const float *x = f.logits + (size_t)b * T * f.V;
                res = accept_warp_small(
                    top_r,
                    [&](int, int pa, int tk) {
                        const float pt = expf(__ldg(x + (size_t)pa * f.V + tk) * f.inv_temp - node_value(lse_r, pa));
                        return pt > fminf(f.epsilon, f.delta * expf(-node_value(ent_r, pa)));
                    },
                    par_b, tok_b, P, T, f.V, p.S_max, lane, path_r);
            } else {
                res = accept_warp_small(
                    top_r, [&](int, int pa, int tk) { return tk == node_value(top_r, pa); }, par_b, tok_b, P,
                    T, f.V, p.S_max, lane, path_r);
            }
            if (designated) {
#pragma unroll
                for (int k = 0; k < 2; ++k)
                    if (lane + 32 * k < T) f.path[(size_t)b * T + lane + 32 * k] = path_r[k];
            }
        } else {
            for (int r = lane; r < T; r += 32) {
                top[r] = row_top(r, s_lse[r], s_ent[r]);
                if (designated) f.argmax_out[(size_t)b * T + r] = top[r];
            }
            __syncwarp();
            const auto top_of = [&](int n) { return top[n]; };
            res = f.typical
                      ? accept_warp_typical(top_of, f.logits + (size_t)b * T * f.V,
                                            [&](int n) { return s_lse[n]; }, [&](int n) { return s_ent[n]; },
                                            f.inv_temp, f.epsilon, f.delta, par_b, tok_b, P, T, f.V, p.S_max,
                                            lane, s_par, path)
                      : accept_warp(top_of, par_b, tok_b, P, T, f.V, p.S_max, lane, s_par, path);
            if (designated)
                for (int i = lane; i < T; i += 32) f.path[(size_t)b * T + i] = path[i];
        }
        if (designated && lane == 0) {
            f.accept_len[b] = res.n_acc;
            f.next_token[b] = res.next_token;
            f.new_prefix_len[b] = res.new_prefix_len;
            atomicMax(f.status + b, res.status);
        }
        if (has_unit && res.n_acc > 0) {
            // cache rows [P_b, P_b + n_acc) <- the accepted tree rows
            const int n = res.n_acc;
            // each slice once: by the CTA holding the first tile of its first query block
            owns_first_tile([&](int u) {
                const int lbh = u / p.n_qb;
                if (u % p.n_qb != 0 || ((lbh / p.H) % B) != b) return false;
                // four 16-byte pieces of K and of V per lane loaded before any is
                // stored, so a slice's rows cost one round trip
                for (int w0 = 0; w0 < n * chunks; w0 += 4 * 32) {
                    uint4 kx[4], vx[4];
                    size_t dof[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int w = w0 + u * 32 + lane;
                        const bool in = w < n * chunks;
                        const int j = in ? w / chunks : 0, c = w - j * chunks;
                        const int src = small ? node_value(path_r, j) : (in ? path[j] : 0);
                        if (in) {
                            const size_t so = ((size_t)lbh * T + src) * f.row_bytes + (size_t)c * 16;
                            dof[u] = ((size_t)lbh * p.S_max + P + j) * f.row_bytes + (size_t)c * 16;
                            kx[u] = __ldg(reinterpret_cast<const uint4 *>(f.k_tree + so));
                            vx[u] = __ldg(reinterpret_cast<const uint4 *>(f.v_tree + so));
                        }
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        if (w0 + u * 32 + lane < n * chunks) {
                            *reinterpret_cast<uint4 *>(f.k_cache + dof[u]) = kx[u];
                            *reinterpret_cast<uint4 *>(f.v_cache + dof[u]) = vx[u];
                        }
                    }
                }
                return false;
            });
        }
        __syncwarp();
    }
}

// Launch one of the persistent attention kernels: one CTA per SM (at most one
// per unit, or with the work split at most one per tile and kSplitMaxGrid) of
// `threads` threads, `smem` bytes of dynamic shared memory, with programmatic
// stream serialization when asked, and as a cooperative launch (all CTAs
// resident at once, or the launch fails) when the fused step's side warps
// compute the argmax in-grid.  The shared-memory opt-in is set once per
// device.
template <class Kern>
cudaError_t launch_attention_grid(Kern kern, uint32_t smem, int threads,
                                  std::atomic<uint64_t> &configured,
                                  const AttnMaps &m, const AttnParams &p, int num_sms,
                                  bool programmatic, cudaStream_t stream)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = dev < 64 ? (1ull << dev) : 0ull;
    if (!bit || !(configured.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        configured.fetch_or(bit, std::memory_order_acq_rel);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)attention_grid(p, num_sms));
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    unsigned n_attr = 0;
    if (programmatic) {
        attr[n_attr].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n_attr].val.programmaticStreamSerializationAllowed = 1;
        ++n_attr;
    }
    if (p.fused && p.fs.in_grid) {
        // the side warps wait for one another's flags: every CTA must be resident
        attr[n_attr].id = cudaLaunchAttributeCooperative;
        attr[n_attr].val.cooperative = 1;
        ++n_attr;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n_attr;
    return cudaLaunchKernelEx(&cfg, kern, m.q, m.kc, m.vc, m.kt, m.vt, p);
}

}  // namespace ppd

