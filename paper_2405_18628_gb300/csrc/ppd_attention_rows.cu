// ppd_attention_rows.cu -- tree-masked attention of the PPD verification step
// for trees of 65..512 tokens on sm_103a (paper Section 3 step (1): tree
// attention over the candidate tree; Section 4.1: every tree token attends to
// the cached prefix, its tree ancestors and itself).
//
// With more than 64 tree tokens the queries fill the tensor core's M side, so
// this kernel keeps one query per TMEM lane (queries zero-padded to 128).  A
// unit is a (layer, sequence, head) slice and a block of 128 of its query rows;
// its tiles are the KV prefix and then the tree's keys, 128 per tile:
//
//   S  = Q * K_tile^T          tcgen05.mma, M = 128 queries, N = 128 keys, K = D
//   P  = exp2(S*scale*log2e - m)   two softmax warps per 32 query rows, each
//                              thread owning one query row and 64 of the 128
//                              keys; P is split into bf16 hi + lo and written
//                              back to TMEM over the scores it came from
//   O += P_hi * V + P_lo * V   tcgen05.mma with A read from TMEM, M = 128
//                              queries, N = D, two products per 16 keys
//
// A row's running maximum and row sum are registers of its two threads; they
// exchange partial maxima through shared memory only on the exact path (a
// unit's first tile, or a score more than 2^16 above the running maximum --
// decided per tile by a vote over the softmax warps) and partial sums at the
// end of a unit.  The tree mask is a 64-bit ancestor bitset per thread, built
// from the parent array in registers.  Three score buffers in TMEM let two PV
// products and the next S product queue in the tensor pipe; the single O
// accumulator of a finished unit is read back after the next unit's first
// tile, and that unit's first PV product waits for the readback.  The unit
// walk (with the work split), the fused step's side warp and the merge of a
// cut unit's partial states are those of the kernel for trees of up to 64
// tokens (ppd_attention.cu), and so are the warp roles (352 threads), except
// that the producer queues each V tile two tiles behind its K tile, the order
// in which the MMA issuer consumes them.
#include "ppd_attention_common.cuh"

#include <cmath>

namespace ppd {

template <int D_>
struct RowsLayout {
    static constexpr int D = D_;
    static constexpr int KT = 128;                         // keys per tile
    static constexpr int M = 128;                          // query rows per unit (zero-padded)
    static constexpr int DCH = D / 64;                     // 64-column groups along D
    static constexpr uint32_t GROUP_BYTES = 128 * 128;     // 128 rows of 64 bf16
    static constexpr uint32_t TILE_BYTES = KT * D * 2;
    static constexpr uint32_t Q_BYTES = M * D * 2;
    static constexpr int QS = 2;                           // Q buffers
    static constexpr int KS = (D == 64) ? 4 : 2;           // K tile ring
    static constexpr int VS = (D == 64) ? 4 : 3;           // V tile ring

    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_K = OFF_Q + QS * Q_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + KS * TILE_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_V + VS * TILE_BYTES;
    static constexpr int B_QFULL = 0;
    static constexpr int B_QEMPTY = B_QFULL + QS;
    static constexpr int B_KFULL = B_QEMPTY + QS;
    static constexpr int B_KEMPTY = B_KFULL + KS;
    static constexpr int B_VFULL = B_KEMPTY + KS;
    static constexpr int B_VEMPTY = B_VFULL + VS;
    // Score tiles in TMEM: P is written over S, so S(g + NSB) waits for PV(g);
    // three buffers keep two PV products and one S product in the tensor pipe.
    static constexpr int NSB = 3;
    static constexpr int B_SFULL = B_VEMPTY + VS;   // [NSB] scores of tile g in TMEM
    static constexpr int B_PFULL = B_SFULL + NSB;   // [NSB] probabilities of tile g in TMEM (8 warps)
    static constexpr int B_PDONE = B_PFULL + NSB;   // [NSB] PV product of tile g complete
    static constexpr int B_OFREE = B_PDONE + NSB;   // a unit's output read back from TMEM (8 warps)
    static constexpr int B_DRAIN = B_OFREE + 1;
    static constexpr int NBAR = B_DRAIN + 1;
    static constexpr uint32_t OFF_TMEMPTR = OFF_BAR + NBAR * 8;
    static constexpr uint32_t OFF_ABORT = OFF_TMEMPTR + 4;
    static constexpr uint32_t OFF_XM = (OFF_ABORT + 4 + 15) & ~15u;   // [2][M] partial row maxima
    static constexpr uint32_t OFF_XL = OFF_XM + 2 * M * 4;            // [2][M] partial row sums
    static constexpr uint32_t OFF_RANGE = OFF_XL + 2 * M * 4;        // WorkRange
    static constexpr uint32_t SMEM_BYTES = OFF_RANGE + ((sizeof(WorkRange) + 15) & ~15u);
    // TMEM columns: S0 | S1 | S2 (128 each; P is written over S) | O (D)
    static constexpr uint32_t T_S = 0, T_O = NSB * 128, TMEM_COLS = 512;
    static_assert(NSB * 128 + D <= 512, "TMEM budget");

    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static_assert((OFF_K | OFF_V | Q_BYTES) % 1024 == 0, "1024-byte aligned operand tiles");
};

template <int D, bool SPLIT>
__global__ void __launch_bounds__(352, 1)
tree_attention_rows_kernel(const __grid_constant__ CUtensorMap map_q,
                           const __grid_constant__ CUtensorMap map_kc,
                           const __grid_constant__ CUtensorMap map_vc,
                           const __grid_constant__ CUtensorMap map_kt,
                           const __grid_constant__ CUtensorMap map_vt, const AttnParams p)
{
    using Lay = RowsLayout<D>;
    extern __shared__ __align__(1024) uint8_t smem[];
    if (smem_addr(smem) & 1023u) {
        if (threadIdx.x == 0 && p.dev_status)
            for (int b = 0; b < p.B; ++b) p.dev_status[b] = kErrUnsupported;
        return;
    }

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Lay::OFF_BAR);
    uint32_t *tmem_ptr = reinterpret_cast<uint32_t *>(smem + Lay::OFF_TMEMPTR);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + Lay::OFF_ABORT);
    float *xm = reinterpret_cast<float *>(smem + Lay::OFF_XM);
    float *xl = reinterpret_cast<float *>(smem + Lay::OFF_XL);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int T = p.T;

    if (threadIdx.x == 0) {
        for (int i = 0; i < Lay::NBAR; ++i)
            mbar_init(bars + i, ((i >= Lay::B_PFULL && i < Lay::B_PFULL + Lay::NSB) || i == Lay::B_OFREE)
                                    ? 8u : 1u);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 9) {
        tmem_alloc(tmem_ptr, Lay::TMEM_COLS);
        tmem_relinquish();
    }
    if (warp == 8 && lane == 0) {
        // the tensor maps are kernel parameters: fetch them before any wait
        tma_prefetch_map(&map_q);
        tma_prefetch_map(&map_kc);
        tma_prefetch_map(&map_vc);
        tma_prefetch_map(&map_kt);
        tma_prefetch_map(&map_vt);
    }
    // in a chain of programmatic launches the inputs may come from the preceding
    // grid: everything above overlapped it, nothing below reads before it is done
    // (the first K/V tiles are only asked of L2 before)
    if (p.pdl_wait) {
        if (warp == 8) prefetch_first_tiles<SPLIT>(p, lane, &map_kc, &map_vc, Lay::DCH, 3);
        asm volatile("griddepcontrol.wait;" ::: "memory");
    }
    WorkRange *wr_s = reinterpret_cast<WorkRange *>(smem + Lay::OFF_RANGE);
    if (warp == 8) {
        const WorkRange w = plan_range(p, lane);   // whole units round-robin without p.split
        if (lane == 0) {
            *wr_s = w;
            if (SPLIT) p.split_rec[blockIdx.x].u = -1;   // no cut unit recorded yet
        }
    }
    // the merge of cut units, or the next call of a chain (a dependent launch),
    // may be scheduled now; it waits for this grid to complete
    if (SPLIT || p.pdl_wait) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_ptr;
    const WorkRange &wr = *wr_s;

    if (warp == 10) {
        // ------------------------------------------------------------ fused-step side work
        if (p.fused) fused_side_warp<false>(p, wr, lane, abort_flag);
    } else if (warp == 8) {
        // ------------------------------------------------------------ TMA producer
        // One queue of copies in the order the MMA issuer consumes them -- S(g)
        // then PV(g - 2) -- so each tile's V follows the K tile two tiles later:
        // Q(unit), K(g), V(g - 2), K(g + 1), V(g - 1), ...  An SM's copies land
        // roughly in issue order, so a V tile queued ahead of its turn would
        // hold back the K tile the next score product waits for, and vice versa.
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            constexpr int LAG = 2;
            int v_row[LAG + 1], v_lbh[LAG + 1];
            bool v_tree[LAG + 1];
            int g = 0, gv = 0, k = 0;
            auto load_v = [&]() {   // V tile gv (its coordinates queued when K(gv) was loaded)
                const int i = gv % (LAG + 1);
                const int vs = gv % Lay::VS;
                if (gv >= Lay::VS)
                    mbar_wait(bars + Lay::B_VEMPTY + vs, ((gv / Lay::VS) - 1) & 1, abort_flag);
                if (!*abort_flag) {
                    mbar_arrive_expect_tx(bars + Lay::B_VFULL + vs, Lay::TILE_BYTES);
#pragma unroll
                    for (int c = 0; c < Lay::DCH; ++c)
                        tma_load_3d(smem + Lay::OFF_V + vs * Lay::TILE_BYTES + c * Lay::GROUP_BYTES,
                                    v_tree[i] ? &map_vt : &map_vc, bars + Lay::B_VFULL + vs, c * 64,
                                    v_row[i], v_lbh[i], pol);
                }
                ++gv;
            };
            SegIter<SPLIT> it(wr);
            for (Seg sg; it.next(p, sg); ++k) {
                const UnitInfo &ui = sg.ui;
                const int qs = k % Lay::QS;
                if (k >= Lay::QS)
                    mbar_wait(bars + Lay::B_QEMPTY + qs, ((k / Lay::QS) - 1) & 1, abort_flag);
                if (!*abort_flag) {
                    // rows T..127 of the box lie beyond the tensor and arrive as zeros
                    mbar_arrive_expect_tx(bars + Lay::B_QFULL + qs, Lay::Q_BYTES);
#pragma unroll
                    for (int c = 0; c < Lay::DCH; ++c)
                        tma_load_3d(smem + Lay::OFF_Q + qs * Lay::Q_BYTES + c * Lay::GROUP_BYTES,
                                    &map_q, bars + Lay::B_QFULL + qs, c * 64, ui.qb * Lay::M,
                                    ui.lbh, pol);
                }
                for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                    const bool tree = (j >= ui.n_pref);
                    const int row = (tree ? j - ui.n_pref : j) * Lay::KT;
                    const int ks = g % Lay::KS;
                    if (g >= Lay::KS)
                        mbar_wait(bars + Lay::B_KEMPTY + ks, ((g / Lay::KS) - 1) & 1, abort_flag);
                    if (!*abort_flag) {
                        mbar_arrive_expect_tx(bars + Lay::B_KFULL + ks, Lay::TILE_BYTES);
#pragma unroll
                        for (int c = 0; c < Lay::DCH; ++c)
                            tma_load_3d(smem + Lay::OFF_K + ks * Lay::TILE_BYTES + c * Lay::GROUP_BYTES,
                                        tree ? &map_kt : &map_kc, bars + Lay::B_KFULL + ks, c * 64,
                                        row, ui.lbh, pol);
                    }
                    const int i = g % (LAG + 1);
                    v_row[i] = row;
                    v_lbh[i] = ui.lbh;
                    v_tree[i] = tree;
                    if (g >= LAG) load_v();
                }
            }
            while (gv < g) load_v();
            if (*abort_flag) {
                // let every copy already issued land before the CTA can exit
                for (int i = max(0, g - Lay::KS); i < g; ++i)
                    mbar_wait_drain(bars + Lay::B_KFULL + i % Lay::KS, (i / Lay::KS) & 1);
                for (int i = max(0, k - Lay::QS); i < k; ++i)
                    mbar_wait_drain(bars + Lay::B_QFULL + i % Lay::QS, (i / Lay::QS) & 1);
                for (int i = max(0, gv - Lay::VS); i < gv; ++i)
                    mbar_wait_drain(bars + Lay::B_VFULL + i % Lay::VS, (i / Lay::VS) & 1);
            }
        }
    } else if (warp == 9) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc_qk = make_idesc_bf16(128, 128, 0, 0);
            const uint32_t idesc_pv = make_idesc_bf16(128, D, 0, 1);
            const uint32_t sq = smem_addr(smem + Lay::OFF_Q);
            const uint32_t sk = smem_addr(smem + Lay::OFF_K);
            const uint32_t sv = smem_addr(smem + Lay::OFF_V);

            // O += P_hi V + P_lo V for tile gp.  Per 32 keys the probability columns
            // hold 8 columns of hi pairs for keys 0..15, 8 for keys 16..31, then the
            // lo pairs in the same order.
            // A unit's first PV product overwrites O: unit k >= 1 waits until the
            // softmax warps have read unit k-1's output back.
            const uint32_t t_o = tmem_base + Lay::T_O;
            auto issue_pv = [&](int gp, bool first, int kp) {
                const int pb = gp % Lay::NSB;
                mbar_wait(bars + Lay::B_PFULL + pb, (gp / Lay::NSB) & 1, abort_flag);
                if (first && kp >= 1) mbar_wait(bars + Lay::B_OFREE, (kp - 1) & 1, abort_flag);
                const int vs = gp % Lay::VS;
                mbar_wait(bars + Lay::B_VFULL + vs, (gp / Lay::VS) & 1, abort_flag);
                tc_fence_after();
                if (!*abort_flag) {
                    const uint32_t a0 = tmem_base + Lay::T_S + (uint32_t)pb * 128u;
                    const uint64_t b0 = make_smem_desc(sv + vs * Lay::TILE_BYTES, Lay::GROUP_BYTES, 1024);
#pragma unroll
                    for (int kk = 0; kk < Lay::KT / 16; ++kk) {
                        const uint64_t b = desc_advance(b0, kk * 2048);
                        const uint32_t a_hi = a0 + 32u * (kk >> 1) + 8u * (kk & 1);
                        umma_bf16_ta(t_o, a_hi, b, idesc_pv, (first && kk == 0) ? 0u : 1u);
                        umma_bf16_ta(t_o, a_hi + 16u, b, idesc_pv, 1u);
                    }
                }
                umma_commit(bars + Lay::B_PDONE + pb);
                umma_commit(bars + Lay::B_VEMPTY + vs);
            };

            // Tiles are issued as S(g), PV(g-2), across unit boundaries: the scores
            // of the tile after next are queued in the tensor pipe before the PV
            // product that has to wait for the softmax of the current tile, so the
            // softmax warps find S(g+1) ready when they finish tile g.  (S(g) reuses
            // the buffer of tile g-3, whose PV product was issued one tile earlier.)
            int g = 0, k = 0;
            int lag_g[2] = {-1, -1}, lag_k[2] = {0, 0};   // tiles g-2 and g-1 awaiting PV
            bool lag_first[2] = {false, false};
            SegIter<SPLIT> it(wr);
            for (Seg sg; it.next(p, sg); ++k) {
                const int qs = k % Lay::QS;
                mbar_wait(bars + Lay::B_QFULL + qs, (k / Lay::QS) & 1, abort_flag);
                for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                    const int ks = g % Lay::KS;
                    const int sb = g % Lay::NSB;
                    mbar_wait(bars + Lay::B_KFULL + ks, (g / Lay::KS) & 1, abort_flag);
                    // P(g - NSB) lives in this S buffer until its PV product is done
                    if (g >= Lay::NSB)
                        mbar_wait(bars + Lay::B_PDONE + sb, ((g - Lay::NSB) / Lay::NSB) & 1, abort_flag);
                    tc_fence_after();
                    if (!*abort_flag) {
                        const uint64_t a0 = make_smem_desc(sq + qs * Lay::Q_BYTES, 16, 1024);
                        const uint64_t b0 = make_smem_desc(sk + ks * Lay::TILE_BYTES, 16, 1024);
                        const uint32_t d_s = tmem_base + Lay::T_S + sb * 128u;
#pragma unroll
                        for (int kk = 0; kk < D / 16; ++kk) {
                            const uint32_t off = (kk >> 2) * Lay::GROUP_BYTES + (kk & 3) * 32;
                            umma_bf16(d_s, desc_advance(a0, off), desc_advance(b0, off), idesc_qk,
                                      kk > 0 ? 1u : 0u);
                        }
                    }
                    umma_commit(bars + Lay::B_SFULL + sb);
                    umma_commit(bars + Lay::B_KEMPTY + ks);
                    if (j == sg.j1 - 1) umma_commit(bars + Lay::B_QEMPTY + qs);
                    if (lag_g[0] >= 0) issue_pv(lag_g[0], lag_first[0], lag_k[0]);
                    lag_g[0] = lag_g[1];
                    lag_first[0] = lag_first[1];
                    lag_k[0] = lag_k[1];
                    lag_g[1] = g;
                    lag_first[1] = (j == sg.j0);
                    lag_k[1] = k;
                }
            }
            for (int x = 0; x < 2; ++x)
                if (lag_g[x] >= 0) issue_pv(lag_g[x], lag_first[x], lag_k[x]);
            umma_commit(bars + Lay::B_DRAIN);
            mbar_wait_drain(bars + Lay::B_DRAIN, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax warps
        const int qd = warp & 3;                 // TMEM lane quadrant of this warp
        const int h = warp >> 2;                 // key half: keys [64h, 64h + 64) of a tile
        const int q = qd * 32 + lane;            // query row (tree token) of this thread
        const uint32_t lane_off = (uint32_t)(qd * 32) << 16;
        const float sl2 = p.scale_log2;
        const bool vec_out = (reinterpret_cast<uintptr_t>(p.out) & 15u) == 0;
        const bool out32 = (reinterpret_cast<uintptr_t>(p.out) & 31u) == 0;

        float m = -INFINITY;    // running maximum of the row (log2 units), same in both threads
        float l = 0.f;          // this thread's share of the row sum
        // anc[t] bit i: tree node 128t + 64h + i is an ancestor of (or is) this
        // thread's query; tmask: the word of the current tree tile
        uint64_t anc[kMaxTree / 128] = {};
        uint64_t tmask = 0;
        int cur_key = -1;
        int g = 0;
        // a finished segment whose output still sits in TMEM; a partial one (a
        // unit cut by the work split) goes to its slot instead of the output
        // pend_f: bit 0 a segment is pending, bit 1 it is partial, bit 2 it was
        // the range's first segment; pend_m, pend_l its row's maximum and sum
        int pend_f = 0, pend_u = 0, pend_g = 0;
        float pend_m = 0.f, pend_l = 0.f;


        // Probabilities of this thread's 64 keys from its raw scores s against the
        // maximum mx (exponents clamped at 64), split into bf16 hi + lo and stored
        // over the scores in TMEM; `lt` gets their sum and `maxd` the largest
        // unclamped exponent.
        auto emit = [&](auto kind_c, const uint32_t (&s)[4][16], float mx, int n_valid,
                        uint32_t t_s, float &lt, float &maxd) {
            constexpr int KIND = decltype(kind_c)::value;
            float lt4[4] = {0.f, 0.f, 0.f, 0.f};
            float md2[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                uint32_t wh[16], wl[16];
#pragma unroll
                for (int e = 0; e < 32; e += 2) {
                    float pv[2];
                    uint32_t hb[2];
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        const int i = 32 * c + e + x;          // key 64h + i of the tile
                        float d = fmaf(__uint_as_float(s[i >> 4][i & 15]), sl2, -mx);
                        if (KIND == kMaskRows) d = (64 * h + i < n_valid) ? d : -INFINITY;
                        if (KIND == kMaskTree) d = ((tmask >> i) & 1ull) ? d : -INFINITY;
                        md2[x] = fmaxf(md2[x], d);
                        pv[x] = ex2(fminf(d, 64.f));
                        lt4[(e >> 1) & 3] += pv[x];
                        hb[x] = __float_as_uint(pv[x]) & 0xFFFF0000u;
                    }
                    wh[e >> 1] = __byte_perm(hb[0], hb[1], 0x7632);
                    const __nv_bfloat162 lo = __floats2bfloat162_rn(pv[0] - __uint_as_float(hb[0]),
                                                                    pv[1] - __uint_as_float(hb[1]));
                    wl[e >> 1] = *reinterpret_cast<const uint32_t *>(&lo);
                }
                tmem_st16(t_s + 32u * c, wh);
                tmem_st16(t_s + 32u * c + 16u, wl);
            }
            lt = (lt4[0] + lt4[1]) + (lt4[2] + lt4[3]);
            maxd = fmaxf(md2[0], md2[1]);
        };

        // Largest visible scaled score among this thread's 64 keys.
        auto part_max = [&](auto kind_c, const uint32_t (&s)[4][16], int n_valid) {
            constexpr int KIND = decltype(kind_c)::value;
            float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                const float v = __uint_as_float(s[i >> 4][i & 15]) * sl2;
                bool vis = true;
                if (KIND == kMaskRows) vis = 64 * h + i < n_valid;
                if (KIND == kMaskTree) vis = ((tmask >> i) & 1ull) != 0;
                mx[i & 3] = fmaxf(mx[i & 3], vis ? v : -INFINITY);
            }
            return fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        };

        // Output of a finished unit: this thread's half of the row of O times 1 / l;
        // then O is free for the next unit's first PV product.
        auto read_back = [&](int lbh_out, int qb_out, int g_last, float linv) {
            mbar_wait(bars + Lay::B_PDONE + g_last % Lay::NSB, (g_last / Lay::NSB) & 1, abort_flag);
            tc_fence_after();
            const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)h * (D / 2);
            const int qg = qb_out * Lay::M + q;
            float *orow = p.out + ((size_t)lbh_out * T + qg) * D + h * (D / 2);
            // the half row in two round trips to TMEM, then full-sector stores
            uint32_t r[2][16];
#pragma unroll
            for (int c2 = 0; c2 < D / 32; c2 += 2) {
#pragma unroll
                for (int ch = 0; ch < 2; ++ch) tmem_ld16(t_o + (c2 + ch) * 16, r[ch]);
                tmem_wait_ld();
                if (qg >= T) continue;
#pragma unroll
                for (int ch = 0; ch < 2; ++ch) {
                    if (out32) {
#pragma unroll
                        for (int e = 0; e < 16; e += 8)
                            st_global_v8(orow + (c2 + ch) * 16 + e, r[ch] + e, linv);
                    } else if (vec_out) {
#pragma unroll
                        for (int e = 0; e < 16; e += 4)
                            *reinterpret_cast<float4 *>(orow + (c2 + ch) * 16 + e) =
                                make_float4(__uint_as_float(r[ch][e]) * linv, __uint_as_float(r[ch][e + 1]) * linv,
                                            __uint_as_float(r[ch][e + 2]) * linv,
                                            __uint_as_float(r[ch][e + 3]) * linv);
                    } else {
#pragma unroll
                        for (int e = 0; e < 16; ++e) orow[(c2 + ch) * 16 + e] = __uint_as_float(r[ch][e]) * linv;
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bars + Lay::B_OFREE);
        };

        // Partial state of a cut unit into slot `slot`: this thread's half of the
        // row of O unnormalised, and (h == 0) the row's maximum and sum; then O
        // is free.  Slots are 256-byte aligned rows of D floats.
        const size_t slot_floats = split_slot_floats(D);
        auto write_partial = [&](int slot, int qb_out, int g_last, float rm, float rl) {
            mbar_wait(bars + Lay::B_PDONE + g_last % Lay::NSB, (g_last / Lay::NSB) & 1, abort_flag);
            tc_fence_after();
            const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)h * (D / 2);
            float *base = p.split_part + (size_t)slot * slot_floats;
            float *orow = base + (size_t)q * D + h * (D / 2);
            const bool live = qb_out * Lay::M + q < T;
            uint32_t r[2][16];
#pragma unroll
            for (int c2 = 0; c2 < D / 32; c2 += 2) {
#pragma unroll
                for (int ch = 0; ch < 2; ++ch) tmem_ld16(t_o + (c2 + ch) * 16, r[ch]);
                tmem_wait_ld();
                if (live) {
#pragma unroll
                    for (int ch = 0; ch < 2; ++ch)
#pragma unroll
                        for (int e = 0; e < 16; e += 8)
                            st_global_v8(orow + (c2 + ch) * 16 + e, r[ch] + e, 1.f);
                }
            }
            if (h == 0 && live) {
                base[(size_t)kSplitRows * D + q] = rm;
                base[(size_t)kSplitRows * D + kSplitRows + q] = rl;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bars + Lay::B_OFREE);
        };

        // The pending segment: a whole unit's output, or a part's state (counted
        // in at the end of the range).
        auto flush_pending = [&]() {
            const int lbh_o = pend_u / p.n_qb, qb_o = pend_u - lbh_o * p.n_qb;
            if (!SPLIT || !(pend_f & 2)) read_back(lbh_o, qb_o, pend_g, rcp(pend_l));
            else write_partial(2 * (int)blockIdx.x + ((pend_f & 4) ? 0 : 1), qb_o, pend_g, pend_m, pend_l);
        };

        int k = 0;
        SegIter<SPLIT> it(wr);
        for (Seg sg; it.next(p, sg); ++k) {
            const UnitInfo &ui = sg.ui;
            const int qg = ui.qb * Lay::M + q;   // this thread's tree token
            if (ui.b * p.n_qb + ui.qb != cur_key) {
                // ancestors of node qg among tree nodes 128t + [64h, 64h + 64)
#pragma unroll
                for (int t = 0; t < kMaxTree / 128; ++t) anc[t] = 0;
                if (qg < T) {
                    bool bad = false;
                    int a = qg;
                    while (true) {
                        if (((a >> 6) & 1) == h) {
#pragma unroll
                            for (int t = 0; t < kMaxTree / 128; ++t)
                                if ((a >> 7) == t) anc[t] |= 1ull << (a & 63);
                        }
                        const int pa = __ldg(p.parent + (size_t)ui.b * T + a);
                        if (a == 0) {
                            bad = (pa != -1);
                            break;
                        }
                        if (pa < 0 || pa >= a) {
                            bad = true;
                            break;
                        }
                        a = pa;
                    }
                    if (bad && h == 0 && p.dev_status) p.dev_status[ui.b] = kErrTree;
                }
                if (qg == 0 && h == 0 && p.dev_status && (ui.P_raw < 0 || ui.P_raw > p.S_max))
                    p.dev_status[ui.b] = kErrCapacity;
                cur_key = ui.b * p.n_qb + ui.qb;
            }

            for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                const bool tree = (j >= ui.n_pref);
                const int n_valid = tree ? T : min(Lay::KT, ui.P - j * Lay::KT);
                if (tree) {
#pragma unroll
                    for (int t = 0; t < kMaxTree / 128; ++t)
                        if (j - ui.n_pref == t) tmask = anc[t];
                }
                const int kind = tree ? kMaskTree : (n_valid < Lay::KT ? kMaskRows : kMaskNone);
                const int sb = g % Lay::NSB;
                mbar_wait(bars + Lay::B_SFULL + sb, (g / Lay::NSB) & 1, abort_flag);
                tc_fence_after();
                const uint32_t t_s = tmem_base + lane_off + Lay::T_S + (uint32_t)sb * 128u +
                                     (uint32_t)h * 64u;
                uint32_t s[4][16];
#pragma unroll
                for (int i = 0; i < 4; ++i) tmem_ld16(t_s + 16u * i, s[i]);
                tmem_wait_ld();

                float lt = 0.f;
                bool exact = (j == sg.j0);
                if (!exact) {
                    // optimistic pass against the current maximum
                    float maxd = -INFINITY;
                    if (kind == kMaskNone) emit(kind_t<kMaskNone>{}, s, m, n_valid, t_s, lt, maxd);
                    else if (kind == kMaskRows) emit(kind_t<kMaskRows>{}, s, m, n_valid, t_s, lt, maxd);
                    else emit(kind_t<kMaskTree>{}, s, m, n_valid, t_s, lt, maxd);
                    exact = named_bar_or(1, 256, maxd > 16.f);
                }
                if (exact) {
                    float pm;
                    if (kind == kMaskNone) pm = part_max(kind_t<kMaskNone>{}, s, n_valid);
                    else if (kind == kMaskRows) pm = part_max(kind_t<kMaskRows>{}, s, n_valid);
                    else pm = part_max(kind_t<kMaskTree>{}, s, n_valid);
                    xm[h * Lay::M + q] = pm;
                    named_bar_sync(1, 256);
                    const float mn = fmaxf(m, fmaxf(xm[q], xm[Lay::M + q]));
                    const float alpha = (mn == m) ? 1.f : ex2(m - mn);
                    if (j > sg.j0) {
                        if (__any_sync(0xffffffffu, alpha != 1.f)) {
                            // rescale this thread's half of the row of O once the PV
                            // product of the previous tile has landed
                            mbar_wait(bars + Lay::B_PDONE + (g - 1) % Lay::NSB,
                                      ((g - 1) / Lay::NSB) & 1, abort_flag);
                            tc_fence_after();
                            const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)h * (D / 2);
#pragma unroll
                            for (int ch = 0; ch < D / 32; ++ch) {
                                uint32_t r[16];
                                tmem_ld16(t_o + ch * 16, r);
                                tmem_wait_ld();
#pragma unroll
                                for (int e = 0; e < 16; ++e)
                                    r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                                tmem_st16(t_o + ch * 16, r);
                            }
                        }
                        l *= alpha;
                    }
                    m = mn;
                    tmem_wait_st();   // optimistic probabilities are overwritten below
                    float unused;
                    if (kind == kMaskNone) emit(kind_t<kMaskNone>{}, s, m, n_valid, t_s, lt, unused);
                    else if (kind == kMaskRows) emit(kind_t<kMaskRows>{}, s, m, n_valid, t_s, lt, unused);
                    else emit(kind_t<kMaskTree>{}, s, m, n_valid, t_s, lt, unused);
                }
                l += lt;

                // V rows of invisible keys in a partial prefix tile may be NaN: zero them
                if (kind == kMaskRows && h == 0) {
                    const int vs = g % Lay::VS;
                    mbar_wait(bars + Lay::B_VFULL + vs, (g / Lay::VS) & 1, abort_flag);
                    if (q >= n_valid) {
                        const uint32_t vrow = smem_addr(smem + Lay::OFF_V + vs * Lay::TILE_BYTES) + q * 128u;
#pragma unroll
                        for (int c = 0; c < Lay::DCH; ++c)
#pragma unroll
                            for (int x = 0; x < 8; ++x)
                                st_shared_v4(vrow + c * Lay::GROUP_BYTES + x * 16, 0u, 0u, 0u, 0u);
                    }
                }
                tmem_wait_st();
                fence_proxy_async_smem();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bars + Lay::B_PFULL + sb);

                // the previous segment's output, once this segment's first tile is on its way
                if (j == sg.j0 && pend_f) {
                    flush_pending();
                    pend_f = 0;
                }

                if (j == sg.j1 - 1) {
                    // ------------------------------------------ segment end: row sum, LSE
                    xl[h * Lay::M + q] = l;
                    named_bar_sync(1, 256);
                    const float L = xl[q] + xl[Lay::M + q];
                    if ((!SPLIT || seg_whole(sg)) && h == 0 && qg < T && p.lse)
                        p.lse[(size_t)ui.lbh * T + qg] = (m + lg2(L)) * 0.69314718055994530942f;
                    pend_u = sg.u;
                    pend_g = g;
                    pend_m = m;
                    pend_l = L;
                    pend_f = 1;
                    if (SPLIT && !seg_whole(sg)) {
                        // a part: slot 2c for the tail range's first segment, 2c + 1 for its last
                        pend_f |= 2 | (sg.u == wr.u_first ? 4 : 0);
                        // the part holding the unit's first tile records it for the merge
                        if (sg.j0 == 0 && threadIdx.x == 0)
                            p.split_rec[blockIdx.x] = SplitRecord{seg_unit_origin(wr, it, sg), wr.n_tail, sg.u, ui.n_tiles};
                    }
                    m = -INFINITY;
                    l = 0.f;
                }
            }
        }
        if (pend_f) flush_pending();
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (*abort_flag && threadIdx.x == 0) {
        for (int b = 0; b < p.B; ++b) {
            if (p.dev_status) p.dev_status[b] = kErrTimeout;
            if (p.fused) atomicMax(p.fs.status + b, (int)kErrTimeout);
        }
    }
    if (warp == 9) tmem_dealloc(tmem_base, Lay::TMEM_COLS);
}

template <int D>
static cudaError_t launch_rows_t(const AttnMaps &m, const AttnParams &p, int num_sms,
                                 bool programmatic, cudaStream_t stream)
{
    static std::atomic<uint64_t> configured[2] = {{0}, {0}};
    if (p.split)
        return launch_attention_grid(tree_attention_rows_kernel<D, true>, RowsLayout<D>::SMEM_BYTES, 352,
                                     configured[1], m, p, num_sms, programmatic, stream);
    return launch_attention_grid(tree_attention_rows_kernel<D, false>, RowsLayout<D>::SMEM_BYTES, 352,
                                 configured[0], m, p, num_sms, programmatic, stream);
}

cudaError_t launch_tree_attention_rows(const AttnMaps &m, const AttnParams &p, int D, int num_sms,
                                       bool programmatic, cudaStream_t stream)
{
    if (D == 128) return launch_rows_t<128>(m, p, num_sms, programmatic, stream);
    return launch_rows_t<64>(m, p, num_sms, programmatic, stream);
}

}  // namespace ppd
