// ppd_attention_common.cuh -- pieces shared by the two tree-attention kernels
// (ppd_attention.cu for trees of up to 64 tokens, ppd_attention_rows.cu for
// 65..128): the unit walk, drain waits, mask kinds and the fused step's side
// warp.
#pragma once

#include "ppd_accept.cuh"
#include "ppd_device.cuh"
#include "ppd_kernels.h"

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

// Side work of the fused verification step, done by one extra warp of every CTA
// while the other warps stream attention.  Once the preceding argmax grid has
// completed (griddepcontrol.wait), for every sequence b this CTA touches -- or
// is designated to report (b mod grid) -- the warp combines the node argmax
// from the partial maxima, decides acceptance, writes the sequence's outputs
// if designated, and copies the accepted tree K/V rows of this CTA's own
// (layer, sequence, head) slices into the cache.  Attention only reads cache
// rows below each prefix, so the copies never race with it.  Scratch (parent
// copies, top-1 tokens, path) lives in a per-CTA slice of the workspace.
PPD_DEV void fused_side_warp(const AttnParams &p, int lane)
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const FusedStep &f = p.fs;
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
        for (int u = blockIdx.x; u < p.n_units && !has_unit; u += gridDim.x)
            has_unit = ((u / p.n_qb / p.H) % B) == b && u % p.n_qb == 0;
        if (!designated && !has_unit) continue;
        for (int r = lane; r < T; r += 32) {
            const size_t base = ((size_t)b * T + r) * S;
            float bv = __ldcg(f.part_val + base);
            int bi = __ldcg(f.part_idx + base);
#pragma unroll 8
            for (int k = 1; k < S; ++k) consider(__ldcg(f.part_val + base + k), __ldcg(f.part_idx + base + k), bv, bi);
            top[r] = bi;
            if (designated) f.argmax_out[(size_t)b * T + r] = bi;
            if (f.typical) stats_finish(combine_stats(f.part_stats, (int64_t)b * T + r, S), s_lse[r], s_ent[r]);
        }
        __syncwarp();
        const auto top_of = [&](int n) { return top[n]; };
        const AcceptResult res =
            f.typical
                ? accept_warp_typical(top_of, f.logits + (size_t)b * T * f.V,
                                      [&](int n) { return s_lse[n]; }, [&](int n) { return s_ent[n]; },
                                      f.inv_temp, f.epsilon, f.delta, p.parent + (size_t)b * T,
                                      f.cand_tokens + (size_t)b * T, __ldg(p.prefix_len + b), T, f.V,
                                      p.S_max, lane, s_par, path)
                : accept_warp(top_of, p.parent + (size_t)b * T, f.cand_tokens + (size_t)b * T,
                              __ldg(p.prefix_len + b), T, f.V, p.S_max, lane, s_par, path);
        if (designated) {
            for (int i = lane; i < T; i += 32) f.path[(size_t)b * T + i] = path[i];
            if (lane == 0) {
                f.accept_len[b] = res.n_acc;
                f.next_token[b] = res.next_token;
                f.new_prefix_len[b] = res.new_prefix_len;
                atomicMax(f.status + b, res.status);
            }
        }
        if (has_unit && res.n_acc > 0) {
            // cache rows [P_b, P_b + n_acc) <- the accepted tree rows
            const int P = __ldg(p.prefix_len + b);
            const int n = res.n_acc;
            // each slice once: by the CTA holding its first query block
            for (int u = blockIdx.x; u < p.n_units; u += gridDim.x) {
                const int lbh = u / p.n_qb;
                if (u % p.n_qb != 0 || ((lbh / p.H) % B) != b) continue;
                for (int w = lane; w < n * chunks; w += 32) {
                    const int j = w / chunks, c = w - j * chunks;
                    const int src = path[j];
                    const size_t so = ((size_t)lbh * T + src) * f.row_bytes + (size_t)c * 16;
                    const size_t dof = ((size_t)lbh * p.S_max + P + j) * f.row_bytes + (size_t)c * 16;
                    const uint4 kx = __ldg(reinterpret_cast<const uint4 *>(f.k_tree + so));
                    const uint4 vx = __ldg(reinterpret_cast<const uint4 *>(f.v_tree + so));
                    *reinterpret_cast<uint4 *>(f.k_cache + dof) = kx;
                    *reinterpret_cast<uint4 *>(f.v_cache + dof) = vx;
                }
            }
        }
        __syncwarp();
    }
}

// Launch one of the persistent attention kernels: one CTA per SM (at most one
// per unit) of `threads` threads, `smem` bytes of dynamic shared memory, with programmatic stream
// serialization when asked.  The shared-memory opt-in is set once per device.
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
    cfg.gridDim = dim3((unsigned)(p.n_units < num_sms ? p.n_units : num_sms));
    cfg.blockDim = dim3((unsigned)threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, m.q, m.kc, m.vc, m.kt, m.vt, p);
}

}  // namespace ppd

