// ppd_attention.cu -- tree-masked attention of the PPD verification step on
// sm_103a (paper Section 3 step (1): tree attention over the candidate tree;
// Section 4.1: every tree token attends to the cached prefix, its tree
// ancestors and itself).
//
// One persistent CTA per SM walks a list of (layer, sequence, head) units.  A
// unit streams its KV prefix in tiles of 128 keys and finishes with one tile
// holding the tree's own keys.  Per tile:
//
//   S^T = K_tile * Q^T     tcgen05.mma, M = 128 keys, N = T_pad queries, K = D
//                          (keys on the M side, so a 64-token tree wastes no
//                          tensor-core rows), accumulated in TMEM
//   P   = exp2(S*scale*log2e - m)   by two softmax warpgroups, one key row per
//                          thread, split into bf16 hi + lo parts (P = hi + lo to
//                          ~2^-16) and written to shared memory
//   O^T += V^T * [P_hi | P_lo]^T    one tcgen05.mma, M = D, N = 2*T_pad, K = 128
//
// Warp roles (352 threads): warps 0-7 softmax (two warpgroups, each owning
// half of the query columns), warp 8 TMA producer, warp 9 MMA issuer and TMEM
// owner, warp 10 the fused step's argmax / acceptance / compaction.  This
// kernel serves trees of up to 64 tokens; larger trees fill the tensor core's
// M side with queries and run the query-row kernel (ppd_attention_rows.cu).
// The running row maximum m is updated lazily: a tile is first done
// with the current m, and only if a score exceeds m by more than 2^16 (or on
// a unit's first tile) does it take the exact path -- a cross-lane maximum,
// a rescale of O and of the row sums, and recomputed probabilities.  The
// tree mask is an ancestor bitset built from the parent array; rows beyond
// the prefix (which may hold anything, NaN included) are masked by select
// and their V rows are zeroed in shared memory before the PV product.  O is
// double-buffered in TMEM and a unit's output is read back only after the
// next unit's first tile, so the stream of tiles never waits for a unit's
// last PV product.  With the work split (ppd_attention_common.cuh) a CTA's
// tiles are an equal share of the launch's; a unit cut by a share boundary is
// done in parts whose partial states the last part merges.
#include "ppd_attention_common.cuh"

#include <cmath>
#include <type_traits>

namespace ppd {

template <int D_>
struct AttnLayout {
    static constexpr int D = D_;
    static constexpr int TPMAX = 64;              // largest padded tree size served
    static constexpr int KT = 128;                // keys per tile
    static constexpr int DCH = D / 64;            // 64-column (128-byte) groups along D
    static constexpr uint32_t GROUP_BYTES = KT * 128;   // one column group of a tile
    static constexpr uint32_t TILE_BYTES = KT * D * 2;
    static constexpr uint32_t Q_GROUP_BYTES = TPMAX * 128;
    static constexpr uint32_t Q_BYTES = TPMAX * D * 2;
    static constexpr int P_GROUPS = 2 * TPMAX / 64;      // [hi | lo] columns / 64
    static constexpr uint32_t P_BYTES = P_GROUPS * GROUP_BYTES;
    static constexpr int OB = 2;                          // O accumulators in TMEM
    static constexpr int QS = 2;                          // Q buffers
    // With D = 128 a tile's probabilities fit exactly in its own K slot, free
    // once S^T = K Q^T is done: no dedicated probability tiles, and the freed
    // shared memory buys a third K and V stage.
    static constexpr bool P_IN_K = (D == 128);
    static constexpr int PS = P_IN_K ? 0 : 2;             // dedicated P tiles
    static constexpr int PB = P_IN_K ? 2 : PS;            // P full/free barrier pairs
    static constexpr int KS = P_IN_K ? 3 : 2;             // K tile ring
    static constexpr int VS = P_IN_K ? 3 : 2;             // V tile ring
    static constexpr int NC_MAX = TPMAX / 2;              // query columns per warpgroup
    static constexpr int ANC_WORDS = TPMAX / 32;          // ancestor bitset words per node

    static constexpr uint32_t OFF_Q = 0;
    static constexpr uint32_t OFF_P = OFF_Q + QS * Q_BYTES;
    static constexpr uint32_t OFF_K = OFF_P + PS * P_BYTES;
    static constexpr uint32_t OFF_V = OFF_K + KS * TILE_BYTES;
    static constexpr uint32_t OFF_BAR = OFF_V + VS * TILE_BYTES;
    // barrier indices
    static constexpr int B_QFULL = 0;
    static constexpr int B_QEMPTY = B_QFULL + QS;
    static constexpr int B_KFULL = B_QEMPTY + QS;
    static constexpr int B_KEMPTY = B_KFULL + KS;
    static constexpr int B_VFULL = B_KEMPTY + KS;
    static constexpr int B_VEMPTY = B_VFULL + VS;
    static constexpr int B_SFULL = B_VEMPTY + VS;
    static constexpr int B_SFREE = B_SFULL + 2;
    static constexpr int B_PFULL = B_SFREE + 2;
    static constexpr int B_PFREE = B_PFULL + PB;
    static constexpr int B_DRAIN = B_PFREE + PB;
    static constexpr int NBAR = B_DRAIN + 1;
    static constexpr uint32_t OFF_TMEMPTR = OFF_BAR + NBAR * 8;
    static constexpr uint32_t OFF_ABORT = OFF_TMEMPTR + 4;
    static constexpr uint32_t OFF_M2 = (OFF_ABORT + 4 + 15) & ~15u;
    static constexpr uint32_t OFF_LINV = OFF_M2 + TPMAX * 4;      // [OB][TPMAX] 1 / row sums (row sums of a partial)
    static constexpr uint32_t OFF_PMX = OFF_LINV + OB * TPMAX * 4;  // [OB][TPMAX] maxima of a partial
    static constexpr uint32_t OFF_UNION = OFF_PMX + OB * TPMAX * 4;
    // union: ancestor bitsets [TPMAX][ANC_WORDS] u32, or reduction scratch [2][4][NC_MAX] f32
    static constexpr uint32_t ANC_BYTES = TPMAX * ANC_WORDS * 4;
    static constexpr uint32_t RED_BYTES = 2 * 4 * NC_MAX * 4;
    static constexpr uint32_t UNION_BYTES = ANC_BYTES > RED_BYTES ? ANC_BYTES : RED_BYTES;
    static constexpr uint32_t OFF_RANGE = (OFF_UNION + UNION_BYTES + 15) & ~15u;   // WorkRange
    static constexpr uint32_t SMEM_BYTES = OFF_RANGE + ((sizeof(WorkRange) + 15) & ~15u);
    // TMEM columns: S0 | S1 | O0 (hi | lo) | O1 (hi | lo)
    static constexpr uint32_t T_S = 0, T_O = 2 * TPMAX;
    static constexpr uint32_t TMEM_COLS = 512;

    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static_assert(!P_IN_K || P_BYTES <= TILE_BYTES, "probability tile fits in a K slot");
    static_assert((OFF_P | OFF_K | OFF_V) % 1024 == 0, "1024-byte aligned operand tiles");
    static_assert((2 + 2 * OB) * TPMAX <= 512, "TMEM budget");
};

// Byte offset (from the shared-memory base) of tile g's probability tile.
template <class Lay>
PPD_DEV uint32_t p_offset(int g)
{
    if (Lay::P_IN_K) return Lay::OFF_K + (uint32_t)(g % Lay::KS) * Lay::TILE_BYTES;
    return Lay::OFF_P + (uint32_t)(g % (Lay::PS > 0 ? Lay::PS : 1)) * Lay::P_BYTES;
}


template <int D, bool SPLIT>
__global__ void __launch_bounds__(352, 1)
tree_attention_kernel(const __grid_constant__ CUtensorMap map_q,
                      const __grid_constant__ CUtensorMap map_kc,
                      const __grid_constant__ CUtensorMap map_vc,
                      const __grid_constant__ CUtensorMap map_kt,
                      const __grid_constant__ CUtensorMap map_vt, const AttnParams p)
{
    using Lay = AttnLayout<D>;
    constexpr int TPMAX = Lay::TPMAX;
    extern __shared__ __align__(1024) uint8_t smem[];
    // The swizzled operand tiles need a 1024-byte aligned base; the check is
    // uniform over the CTA, before any barrier.
    if (smem_addr(smem) & 1023u) {
        if (threadIdx.x == 0 && p.dev_status)
            for (int b = 0; b < p.B; ++b) p.dev_status[b] = kErrUnsupported;
        return;
    }

    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Lay::OFF_BAR);
    uint32_t *tmem_ptr = reinterpret_cast<uint32_t *>(smem + Lay::OFF_TMEMPTR);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + Lay::OFF_ABORT);
    float *m2 = reinterpret_cast<float *>(smem + Lay::OFF_M2);
    uint32_t *anc = reinterpret_cast<uint32_t *>(smem + Lay::OFF_UNION);   // [TPMAX][ANC_WORDS]
    float *red = reinterpret_cast<float *>(smem + Lay::OFF_UNION);         // [2][4][NC_MAX]

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int T = p.T;
    const int T_pad = p.T_pad;

    if (threadIdx.x == 0) {
        for (int i = 0; i < Lay::NBAR; ++i) {
            uint32_t count = 1;
            if ((i >= Lay::B_SFREE && i < Lay::B_SFREE + 2) ||
                (i >= Lay::B_PFULL && i < Lay::B_PFULL + Lay::PB))
                count = 8;
            mbar_init(bars + i, count);
        }
        *abort_flag = 0;
        mbar_fence_init();
    }
    for (int i = threadIdx.x; i < TPMAX; i += blockDim.x) m2[i] = -INFINITY;
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
        if (p.fused) fused_side_warp<true>(p, wr, lane, abort_flag);
    } else if (warp == 8) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_first();
            const uint32_t q_tx = (uint32_t)T_pad * 128u * Lay::DCH;
            int g = 0, k = 0;
            SegIter<SPLIT> it(wr);
            for (Seg sg; it.next(p, sg); ++k) {
                const UnitInfo &ui = sg.ui;
                const int u = sg.u;
                const int qs = k % Lay::QS;
                if (k >= Lay::QS)
                    mbar_wait(bars + Lay::B_QEMPTY + qs, ((k / Lay::QS) - 1) & 1, abort_flag);
                if (!*abort_flag) {
                    mbar_arrive_expect_tx(bars + Lay::B_QFULL + qs, q_tx);
#pragma unroll
                    for (int c = 0; c < Lay::DCH; ++c)
                        tma_load_3d(smem + Lay::OFF_Q + qs * Lay::Q_BYTES + c * Lay::Q_GROUP_BYTES,
                                    &map_q, bars + Lay::B_QFULL + qs, c * 64, 0, u, pol);
                }
                for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                    const bool tree = (j == ui.n_pref);
                    const int row = tree ? 0 : j * Lay::KT;
                    const int ks = g % Lay::KS;
                    if (g >= Lay::KS)
                        mbar_wait(bars + Lay::B_KEMPTY + ks, ((g / Lay::KS) - 1) & 1, abort_flag);
                    if (!*abort_flag) {
                        mbar_arrive_expect_tx(bars + Lay::B_KFULL + ks, Lay::TILE_BYTES);
#pragma unroll
                        for (int c = 0; c < Lay::DCH; ++c)
                            tma_load_3d(smem + Lay::OFF_K + ks * Lay::TILE_BYTES + c * Lay::GROUP_BYTES,
                                        tree ? &map_kt : &map_kc, bars + Lay::B_KFULL + ks, c * 64,
                                        row, u, pol);
                    }
                    const int vs = g % Lay::VS;
                    if (g >= Lay::VS)
                        mbar_wait(bars + Lay::B_VEMPTY + vs, ((g / Lay::VS) - 1) & 1, abort_flag);
                    if (!*abort_flag) {
                        mbar_arrive_expect_tx(bars + Lay::B_VFULL + vs, Lay::TILE_BYTES);
#pragma unroll
                        for (int c = 0; c < Lay::DCH; ++c)
                            tma_load_3d(smem + Lay::OFF_V + vs * Lay::TILE_BYTES + c * Lay::GROUP_BYTES,
                                        tree ? &map_vt : &map_vc, bars + Lay::B_VFULL + vs, c * 64,
                                        row, u, pol);
                    }
                }
            }
            if (*abort_flag) {
                // let every copy already issued land before the CTA can exit
                for (int i = max(0, g - Lay::KS); i < g; ++i)
                    mbar_wait_drain(bars + Lay::B_KFULL + i % Lay::KS, (i / Lay::KS) & 1);
                for (int i = max(0, g - Lay::VS); i < g; ++i)
                    mbar_wait_drain(bars + Lay::B_VFULL + i % Lay::VS, (i / Lay::VS) & 1);
                for (int i = max(0, k - Lay::QS); i < k; ++i)
                    mbar_wait_drain(bars + Lay::B_QFULL + i % Lay::QS, (i / Lay::QS) & 1);
            }
        }
    } else if (warp == 9) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc_qk = make_idesc_bf16(128, T_pad, 0, 0);
            const uint32_t idesc_pv = make_idesc_bf16(128, 2 * T_pad, 1, 1);
            const uint32_t sq = smem_addr(smem + Lay::OFF_Q);
            const uint32_t sk = smem_addr(smem + Lay::OFF_K);
            const uint32_t sv = smem_addr(smem + Lay::OFF_V);
            const uint32_t s0 = smem_addr(smem);
            // V^T as the A operand: M = D spans the tile's 64-column groups.  With
            // D = 64 both M halves read the same group (rows 64..127 of O^T repeat
            // rows 0..63 and are ignored).
            const uint32_t v_lbo = (D == 128) ? Lay::GROUP_BYTES : 0u;

            auto issue_pv = [&](int gp, bool first, uint32_t t_o) {
                const int ps = gp % Lay::PB;
                mbar_wait(bars + Lay::B_PFULL + ps, (gp / Lay::PB) & 1, abort_flag);
                const int vs = gp % Lay::VS;
                mbar_wait(bars + Lay::B_VFULL + vs, (gp / Lay::VS) & 1, abort_flag);
                tc_fence_after();
                if (!*abort_flag) {
                    // descriptors built once; each 16-key step moves 2048 bytes on
                    const uint64_t a0 = make_smem_desc(sv + vs * Lay::TILE_BYTES, v_lbo, 1024);
                    const uint64_t b0 = make_smem_desc(s0 + p_offset<Lay>(gp), Lay::GROUP_BYTES, 1024);
#pragma unroll
                    for (int kk = 0; kk < Lay::KT / 16; ++kk)
                        umma_bf16(t_o, desc_advance(a0, kk * 2048), desc_advance(b0, kk * 2048), idesc_pv,
                                  (first && kk == 0) ? 0u : 1u);
                }
                umma_commit(bars + Lay::B_PFREE + ps);
                umma_commit(bars + Lay::B_VEMPTY + vs);
                if (Lay::P_IN_K) umma_commit(bars + Lay::B_KEMPTY + gp % Lay::KS);
            };

            // Tiles are issued as S(g), PV(g-1) across unit boundaries, so the next
            // unit's first scores are under way before this unit's last PV product.
            int g = 0, k = 0;
            int prev_g = -1;
            bool prev_first = false;
            uint32_t prev_to = 0;
            SegIter<SPLIT> it(wr);
            for (Seg sg; it.next(p, sg); ++k) {
                const int qs = k % Lay::QS;
                const uint32_t t_o = tmem_base + Lay::T_O + (uint32_t)(k % Lay::OB) * 2 * TPMAX;
                mbar_wait(bars + Lay::B_QFULL + qs, (k / Lay::QS) & 1, abort_flag);
                for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                    const int ks = g % Lay::KS;
                    const int sb = g & 1;
                    mbar_wait(bars + Lay::B_KFULL + ks, (g / Lay::KS) & 1, abort_flag);
                    if (g >= 2) mbar_wait(bars + Lay::B_SFREE + sb, ((g >> 1) - 1) & 1, abort_flag);
                    tc_fence_after();
                    if (!*abort_flag) {
                        const uint64_t a0 = make_smem_desc(sk + ks * Lay::TILE_BYTES, 16, 1024);
                        const uint64_t b0 = make_smem_desc(sq + qs * Lay::Q_BYTES, 16, 1024);
                        const uint32_t d_s = tmem_base + Lay::T_S + sb * TPMAX;
#pragma unroll
                        for (int kk = 0; kk < D / 16; ++kk) {
                            const uint32_t koff = (kk >> 2) * Lay::GROUP_BYTES + (kk & 3) * 32;
                            const uint32_t qoff = (kk >> 2) * Lay::Q_GROUP_BYTES + (kk & 3) * 32;
                            umma_bf16(d_s, desc_advance(a0, koff), desc_advance(b0, qoff), idesc_qk,
                                      kk > 0 ? 1u : 0u);
                        }
                    }
                    umma_commit(bars + Lay::B_SFULL + sb);
                    if (!Lay::P_IN_K) umma_commit(bars + Lay::B_KEMPTY + ks);
                    if (j == sg.j1 - 1) umma_commit(bars + Lay::B_QEMPTY + qs);
                    if (prev_g >= 0) issue_pv(prev_g, prev_first, prev_to);
                    prev_g = g;
                    prev_first = (j == sg.j0);
                    prev_to = t_o;
                }
            }
            if (prev_g >= 0) issue_pv(prev_g, prev_first, prev_to);
            // all MMAs finished before TMEM can be released
            umma_commit(bars + Lay::B_DRAIN);
            mbar_wait_drain(bars + Lay::B_DRAIN, 0);
        }
    } else {
        // ------------------------------------------------------------ softmax warpgroups
        const int wg = warp >> 2;
        const int wq = warp & 3;
        const int t = wq * 32 + lane;           // key row of S^T, and d of O^T
        const int NC = T_pad >> 1;              // query columns owned by this warpgroup
        const int q0 = wg * NC;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        // this thread's row of the probability tile (128-byte swizzled atoms)
        const uint32_t p_row = smem_addr(smem) + (uint32_t)(t >> 3) * 1024u +
                               (uint32_t)(t & 7) * 128u;
        const uint32_t p_swz = (uint32_t)(t & 7);
        const float sl2 = p.scale_log2;
        float *red_wg = red + wg * 4 * Lay::NC_MAX;
        float *linv = reinterpret_cast<float *>(smem + Lay::OFF_LINV);   // [OB][TPMAX]
        float *pmx = reinterpret_cast<float *>(smem + Lay::OFF_PMX);     // [OB][TPMAX]

        constexpr int NL = Lay::NC_MAX;
        float lacc[NL];   // this key row's share of every owned query's row sum
#pragma unroll
        for (int c = 0; c < NL; ++c) lacc[c] = 0.f;
        uint64_t dbits = 0;   // bit c: key t (tree node t) is visible to query q0 + c
        int cur_b = -1;
        int g = 0;
        int cur_k = 0;        // this CTA's unit counter (selects the O accumulator)
        // a finished segment whose output still sits in TMEM; a partial one (a
        // unit cut by the work split) goes to its slot instead of the output
        // pend_f: bit 0 a segment is pending, bit 1 it is partial, bit 2 it was
        // the range's first segment, bit 3 its O accumulator
        int pend_f = 0, pend_u = 0, pend_g = 0;


        // Probabilities of the 16 query columns [cb, cb+16) of this thread's key row
        // from its raw scores r, against the current running maxima, exponents
        // clamped at 64 so nothing overflows before a rescale.  STORE: split into
        // bf16 hi + lo, store into probability tile `pbuf` (byte offset) and add to
        // lacc.  UNDO: subtract the same values from lacc again (bit-identical to
        // an earlier STORE with the same maxima).  `maxd` collects the largest
        // unclamped exponent.  WAIT: r is the target of a TMEM load still in flight.
        auto emit_half = [&](auto kind_c, auto undo_c, auto wait_c, const uint32_t (&r)[16], int cb,
                             uint32_t bits16, bool row_ok, uint32_t pbuf, float &maxd) {
            constexpr int KIND = decltype(kind_c)::value;
            constexpr bool UNDO = decltype(undo_c)::value != 0;
            const float4 *m4 = reinterpret_cast<const float4 *>(m2 + q0 + cb);
            float m[16];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float4 v = m4[k];
                m[4 * k] = v.x;
                m[4 * k + 1] = v.y;
                m[4 * k + 2] = v.z;
                m[4 * k + 3] = v.w;
            }
            if (decltype(wait_c)::value) tmem_wait_ld();
            float pv[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                float d = fmaf(__uint_as_float(r[e]), sl2, -m[e]);
                if (KIND == kMaskRows) d = row_ok ? d : -INFINITY;
                if (KIND == kMaskTree) d = ((bits16 >> e) & 1u) ? d : -INFINITY;
                maxd = fmaxf(maxd, d);
                pv[e] = ex2(fminf(d, 64.f));
                if (UNDO) lacc[cb + e] -= pv[e];
                else lacc[cb + e] += pv[e];
            }
            if (!UNDO) {
                uint32_t hw[8], lw[8];
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const uint32_t h0 = __float_as_uint(pv[e]) & 0xFFFF0000u;
                    const uint32_t h1 = __float_as_uint(pv[e + 1]) & 0xFFFF0000u;
                    hw[e >> 1] = __byte_perm(h0, h1, 0x7632);
                    const __nv_bfloat162 lo = __floats2bfloat162_rn(pv[e] - __uint_as_float(h0),
                                                                    pv[e + 1] - __uint_as_float(h1));
                    lw[e >> 1] = *reinterpret_cast<const uint32_t *>(&lo);
                }
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    const int ch = q0 + cb + half * 8;   // hi column
                    const int cl = T_pad + ch;            // lo column
                    const uint32_t ah = p_row + pbuf + (uint32_t)(ch >> 6) * Lay::GROUP_BYTES +
                                        ((((uint32_t)(ch & 63) >> 3) ^ p_swz) << 4);
                    const uint32_t al = p_row + pbuf + (uint32_t)(cl >> 6) * Lay::GROUP_BYTES +
                                        ((((uint32_t)(cl & 63) >> 3) ^ p_swz) << 4);
                    st_shared_v4(ah, hw[half * 4], hw[half * 4 + 1], hw[half * 4 + 2], hw[half * 4 + 3]);
                    st_shared_v4(al, lw[half * 4], lw[half * 4 + 1], lw[half * 4 + 2], lw[half * 4 + 3]);
                }
            }
        };
        using store_t = kind_t<0>;
        using undo_t = kind_t<1>;
        using wait_t = kind_t<1>;
        using nowait_t = kind_t<0>;

        // Optimistic pass over query columns [c0, c0+16) (and [c0+16, c0+32) when
        // `two`): scores straight from TMEM against the current maxima.
        auto p_group = [&](auto kind_c, uint32_t t_s, int c0, bool two, bool row_ok, uint32_t pbuf,
                           float &maxd) {
            const uint32_t bits = (uint32_t)(dbits >> c0);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (h == 0 || two) {
                    uint32_t r[16];
                    tmem_ld16(t_s + c0 + h * 16, r);
                    emit_half(kind_c, store_t{}, wait_t{}, r, c0 + h * 16, bits >> (h * 16), row_ok,
                              pbuf, maxd);
                }
            }
        };

        // Exact pass over the same columns, on a unit's first tile or after a score
        // jumped past its maximum: the scores are loaded once and kept in registers;
        // the optimistic contributions are taken back out of the row sums (later
        // tiles); every column's maximum over the 128 key rows is a warp max
        // (redux) combined across the four warps; O and the row sums are rescaled
        // (later tiles); the probabilities are recomputed.
        auto exact_group = [&](auto kind_c, uint32_t t_s, int c0, bool two, bool row_ok,
                               uint32_t pbuf, bool later, bool &o_ready) {
            constexpr int KIND = decltype(kind_c)::value;
            uint32_t r0[16], r1[16];
            tmem_ld16(t_s + c0, r0);
            if (two) tmem_ld16(t_s + c0 + 16, r1);
            tmem_wait_ld();
            const uint32_t bits = (uint32_t)(dbits >> c0);
            if (later) {
                float unused = 0.f;
                emit_half(kind_c, undo_t{}, nowait_t{}, r0, c0, bits, row_ok, pbuf, unused);
                if (two) emit_half(kind_c, undo_t{}, nowait_t{}, r1, c0 + 16, bits >> 16, row_ok, pbuf, unused);
            }
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                if (e < 16 || two) {
                    const float sv = __uint_as_float(e < 16 ? r0[e] : r1[e - 16]);
                    const bool vis = KIND == kMaskNone ? true
                                     : KIND == kMaskRows ? row_ok
                                                         : ((bits >> e) & 1u) != 0;
                    const float mx = warp_max(vis ? sv * sl2 : -INFINITY);
                    if (lane == e) red_wg[wq * Lay::NC_MAX + c0 + e] = mx;
                }
            }
            named_bar_sync(1 + wg, 128);
            const int gw = two ? 32 : 16;
            if (t < gw) {
                const int c = c0 + t;
                const float tm = fmaxf(fmaxf(red_wg[c], red_wg[Lay::NC_MAX + c]),
                                       fmaxf(red_wg[2 * Lay::NC_MAX + c], red_wg[3 * Lay::NC_MAX + c]));
                const float old = m2[q0 + c];
                const float nw = fmaxf(old, tm);
                m2[q0 + c] = nw;
                red_wg[c] = (nw == old) ? 1.f : ex2(old - nw);   // alpha
            }
            named_bar_sync(1 + wg, 128);
            if (later) {
                // rescale the accumulated output columns and row sums; the PV product
                // of the previous tile must have landed first
                if (!o_ready) {
                    const int pp = (g - 1) % Lay::PB;
                    mbar_wait(bars + Lay::B_PFREE + pp, ((g - 1) / Lay::PB) & 1, abort_flag);
                    o_ready = true;
                }
                tc_fence_after();
                const uint32_t t_o = tmem_base + lane_off + Lay::T_O +
                                     (uint32_t)(cur_k % Lay::OB) * 2 * TPMAX;
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    if (h == 0 || two) {
                        const int cb = c0 + h * 16;
                        float a[16];
#pragma unroll
                        for (int e = 0; e < 16; ++e) a[e] = red_wg[cb + e];
#pragma unroll
                        for (int part = 0; part < 2; ++part) {
                            const uint32_t col = t_o + (part ? T_pad : 0) + q0 + cb;
                            uint32_t rr[16];
                            tmem_ld16(col, rr);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 16; ++e)
                                rr[e] = __float_as_uint(__uint_as_float(rr[e]) * a[e]);
                            tmem_st16(col, rr);
                        }
#pragma unroll
                        for (int e = 0; e < 16; ++e) lacc[cb + e] *= a[e];
                    }
                }
                tmem_wait_st();
            }
            float maxd = -INFINITY;
            emit_half(kind_c, store_t{}, nowait_t{}, r0, c0, bits, row_ok, pbuf, maxd);
            if (two) emit_half(kind_c, store_t{}, nowait_t{}, r1, c0 + 16, bits >> 16, row_ok, pbuf, maxd);
        };

        // Output of a finished unit: O (hi + lo) from its TMEM accumulator times the
        // reciprocal row sums, one head-dim element per thread, queries in order.
        auto read_back = [&](int u_out, int ob, int g_last) {
            mbar_wait(bars + Lay::B_PFREE + g_last % Lay::PB, (g_last / Lay::PB) & 1, abort_flag);
            tc_fence_after();
            if (wq * 32 < D) {
                const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)ob * 2 * TPMAX;
                const float *li = linv + ob * TPMAX;
                float *orow = p.out + (size_t)u_out * T * D + t;
#pragma unroll
                for (int ch = 0; ch < Lay::NC_MAX / 16; ++ch) {
                    if (ch * 16 < NC) {
                        uint32_t rh[16], rl[16];
                        tmem_ld16(t_o + q0 + ch * 16, rh);
                        tmem_ld16(t_o + T_pad + q0 + ch * 16, rl);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int q = q0 + ch * 16 + e;
                            if (q < T)
                                orow[(size_t)q * D] =
                                    (__uint_as_float(rh[e]) + __uint_as_float(rl[e])) * li[q];
                        }
                    }
                }
            }
            tc_fence_before();
        };

        // Partial state of a cut unit into slot `slot`: O (hi + lo) unnormalised,
        // each query's running maximum and row sum.
        const size_t slot_floats = split_slot_floats(D);
        auto write_partial = [&](int slot, int ob, int g_last) {
            mbar_wait(bars + Lay::B_PFREE + g_last % Lay::PB, (g_last / Lay::PB) & 1, abort_flag);
            tc_fence_after();
            float *base = p.split_part + (size_t)slot * slot_floats;
            if (wq * 32 < D) {
                const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)ob * 2 * TPMAX;
#pragma unroll
                for (int ch = 0; ch < Lay::NC_MAX / 16; ++ch) {
                    if (ch * 16 < NC) {
                        uint32_t rh[16], rl[16];
                        tmem_ld16(t_o + q0 + ch * 16, rh);
                        tmem_ld16(t_o + T_pad + q0 + ch * 16, rl);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            const int q = q0 + ch * 16 + e;
                            if (q < T) base[(size_t)q * D + t] = __uint_as_float(rh[e]) + __uint_as_float(rl[e]);
                        }
                    }
                }
            }
            if (t < NC && q0 + t < T) {
                base[(size_t)kSplitRows * D + q0 + t] = pmx[ob * TPMAX + q0 + t];
                base[(size_t)kSplitRows * D + kSplitRows + q0 + t] = linv[ob * TPMAX + q0 + t];
            }
            tc_fence_before();
        };

        // The pending segment: a whole unit's output, or a part's state (counted
        // in at the end of the range).
        auto flush_pending = [&]() {
            const int pend_ob = (pend_f >> 3) & 1;
            if (!SPLIT || !(pend_f & 2)) read_back(pend_u, pend_ob, pend_g);
            else write_partial(2 * (int)blockIdx.x + ((pend_f & 4) ? 0 : 1), pend_ob, pend_g);
        };

        int k = 0;
        SegIter<SPLIT> it(wr);
        for (Seg sg; it.next(p, sg); ++k) {
            const UnitInfo &ui = sg.ui;
            const int u = sg.u;
            cur_k = k;
            const int ob = k % Lay::OB;
            const uint32_t t_o = tmem_base + lane_off + Lay::T_O + (uint32_t)ob * 2 * TPMAX;
            if (ui.b != cur_b) {
                // ancestor bitsets of this sequence's tree, one node per thread
                named_bar_sync(3, 256);
                const int i = wg * 128 + t;
                if (i < T) {
                    uint32_t w[Lay::ANC_WORDS];
#pragma unroll
                    for (int x = 0; x < Lay::ANC_WORDS; ++x) w[x] = 0u;
                    bool bad = false;
                    int a = i;
                    while (true) {
#pragma unroll
                        for (int x = 0; x < Lay::ANC_WORDS; ++x)
                            if ((a >> 5) == x) w[x] |= 1u << (a & 31);
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
#pragma unroll
                    for (int x = 0; x < Lay::ANC_WORDS; ++x) anc[i * Lay::ANC_WORDS + x] = w[x];
                    if (bad && p.dev_status) p.dev_status[ui.b] = kErrTree;
                }
                if (i == 0 && p.dev_status && (ui.P_raw < 0 || ui.P_raw > p.S_max))
                    p.dev_status[ui.b] = kErrCapacity;
                named_bar_sync(3, 256);
                dbits = 0;
                if (t < T) {
                    for (int c = 0; c < NC; ++c) {
                        const int q = q0 + c;
                        if (q < T && ((anc[q * Lay::ANC_WORDS + (t >> 5)] >> (t & 31)) & 1u))
                            dbits |= 1ull << c;
                    }
                }
                named_bar_sync(3, 256);
                cur_b = ui.b;
            }

            for (int j = sg.j0; j < sg.j1; ++j, ++g) {
                const bool tree = (j == ui.n_pref);
                const int n_valid = tree ? T : min(Lay::KT, ui.P - j * Lay::KT);
                const bool row_ok = t < n_valid;
                const int kind = tree ? kMaskTree : (n_valid < Lay::KT ? kMaskRows : kMaskNone);
                const int sb = g & 1;
                mbar_wait(bars + Lay::B_SFULL + sb, (g >> 1) & 1, abort_flag);
                tc_fence_after();
                const uint32_t t_s = tmem_base + lane_off + Lay::T_S + sb * TPMAX + q0;
                const int ps = g % Lay::PB;
                const uint32_t pbuf = p_offset<Lay>(g);
                // a dedicated probability tile is free once the PV product of tile
                // g - PS is done; a K slot is free as soon as S(g) is (waited above)
                if constexpr (!Lay::P_IN_K) {
                    if (g >= Lay::PS)
                        mbar_wait(bars + Lay::B_PFREE + ps, ((g / Lay::PS) - 1) & 1, abort_flag);
                }
                bool o_ready = false;   // PV of tile g-1 known to be complete

                // Column groups of up to 32 queries, done optimistically with the
                // current running maxima; on a unit's first tile, or when a score
                // exceeds its maximum by more than 2^16, the group takes the exact
                // path: cross-lane tile maximum, rescale of O and of the row sums,
                // probabilities recomputed.
#pragma unroll
                for (int gc0 = 0; gc0 < Lay::NC_MAX; gc0 += 32) {
                    if (gc0 < NC) {
                        const bool two = gc0 + 16 < NC;
                        bool exact;
                        if (j > sg.j0) {
                            float maxd = -INFINITY;
                            if (kind == kMaskNone) p_group(kind_t<kMaskNone>{}, t_s, gc0, two, row_ok, pbuf, maxd);
                            else if (kind == kMaskRows) p_group(kind_t<kMaskRows>{}, t_s, gc0, two, row_ok, pbuf, maxd);
                            else p_group(kind_t<kMaskTree>{}, t_s, gc0, two, row_ok, pbuf, maxd);
                            exact = named_bar_or(1 + wg, 128, maxd > 16.f);
                        } else {
                            named_bar_sync(1 + wg, 128);   // earlier readers of red_wg are done
                            exact = true;
                        }
                        if (exact) {
                            const bool later = j > sg.j0;
                            if (kind == kMaskNone) exact_group(kind_t<kMaskNone>{}, t_s, gc0, two, row_ok, pbuf, later, o_ready);
                            else if (kind == kMaskRows) exact_group(kind_t<kMaskRows>{}, t_s, gc0, two, row_ok, pbuf, later, o_ready);
                            else exact_group(kind_t<kMaskTree>{}, t_s, gc0, two, row_ok, pbuf, later, o_ready);
                        }
                    }
                }

                // V rows of invisible keys in a partial prefix tile may be NaN: zero them
                if (kind == kMaskRows && wg == 0) {
                    const int vs = g % Lay::VS;
                    mbar_wait(bars + Lay::B_VFULL + vs, (g / Lay::VS) & 1, abort_flag);
                    if (!row_ok) {
                        const uint32_t vrow = smem_addr(smem + Lay::OFF_V + vs * Lay::TILE_BYTES) + t * 128u;
#pragma unroll
                        for (int c = 0; c < Lay::DCH; ++c)
#pragma unroll
                            for (int x = 0; x < 8; ++x)
                                st_shared_v4(vrow + c * Lay::GROUP_BYTES + x * 16, 0u, 0u, 0u, 0u);
                    }
                }
                fence_proxy_async_smem();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(bars + Lay::B_PFULL + ps);
                    mbar_arrive(bars + Lay::B_SFREE + sb);
                }

                // the previous segment's output, once this segment's first tile is on its way
                if (j == sg.j0 && pend_f) {
                    flush_pending();
                    pend_f = 0;
                }

                if (j == sg.j1 - 1) {
                    // ------------------------------------------ unit end: row sums, LSE
                    named_bar_sync(1 + wg, 128);   // every thread is done reading alpha
#pragma unroll
                    for (int ch = 0; ch < Lay::NC_MAX / 16; ++ch) {
                        if (ch * 16 < NC) {
                            float v[16];
#pragma unroll
                            for (int e = 0; e < 16; ++e) v[e] = lacc[ch * 16 + e];
                            const float s = warp_transpose_reduce16(v, lane, OpAdd());
                            if (!(lane & 1)) red_wg[wq * Lay::NC_MAX + ch * 16 + (lane >> 1)] = s;
                        }
                    }
                    named_bar_sync(1 + wg, 128);
                    if (t < NC) {
                        const float l = red_wg[t] + red_wg[Lay::NC_MAX + t] +
                                        red_wg[2 * Lay::NC_MAX + t] + red_wg[3 * Lay::NC_MAX + t];
                        const int q = q0 + t;
                        if (!SPLIT || seg_whole(sg)) {
                            if (p.lse && q < T)
                                p.lse[(size_t)u * T + q] = (m2[q] + lg2(l)) * 0.69314718055994530942f;
                            linv[ob * TPMAX + q] = rcp(l);
                        } else {
                            linv[ob * TPMAX + q] = l;
                            pmx[ob * TPMAX + q] = m2[q];
                        }
                        m2[q] = -INFINITY;
                    }
#pragma unroll
                    for (int c = 0; c < NL; ++c) lacc[c] = 0.f;
                    pend_u = u;
                    pend_g = g;
                    pend_f = 1 | (ob << 3);
                    if (SPLIT && !seg_whole(sg)) {
                        // a part: slot 2c for the tail range's first segment, 2c + 1 for its last
                        pend_f |= 2 | (sg.u == wr.u_first ? 4 : 0);
                        // the part holding the unit's first tile records it for the merge
                        if (sg.j0 == 0 && threadIdx.x == 0)
                            p.split_rec[blockIdx.x] = SplitRecord{seg_unit_origin(wr, it, sg), wr.n_tail, u, ui.n_tiles};
                    }
                }
            }
        }
        if (pend_f) {
            named_bar_sync(1 + wg, 128);   // the row sums are in shared memory
            flush_pending();
        }
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

// The merge of the units cut by the work split: blockIdx.x is an attention
// CTA (gridDim.x = the attention grid), blockIdx.y a block of 256 / (D / 8)
// rows of the unit that CTA recorded; each thread merges 8 columns of a row,
// once the attention grid has completed.
__global__ void __launch_bounds__(256) split_merge_kernel(const AttnParams p, int D)
{
    // a next grid launched as a programmatic dependent may start at once; it
    // waits for this grid to complete before it reads or writes anything
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const SplitRecord r = p.split_rec[blockIdx.x];
    if (r.u < 0) return;
    const int per_row = D / 8;
    const int rows_per_block = (int)blockDim.x / per_row;
    const int lbh = r.u / p.n_qb, qb = r.u - lbh * p.n_qb;
    const int n_rows = min(kSplitRows, p.T - qb * kSplitRows);
    const int row = (int)blockIdx.y * rows_per_block + (int)threadIdx.x / per_row;
    if (row >= n_rows) return;
    const SplitParts sp = split_parts(r.n_tail, r.off, r.n_tiles);
    split_merge_chunk(p.split_part, p.out, p.lse, sp, r.n_tail, (int)gridDim.x,
                      (size_t)lbh * p.T + (size_t)qb * kSplitRows, row, ((int)threadIdx.x % per_row) * 8, D);
}

cudaError_t launch_split_merge(const AttnParams &p, int D, int grid, cudaStream_t stream)
{
    const int rows_per_block = 256 / (D / 8);
    const int rows = p.T < kSplitRows ? p.T : kSplitRows;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid, (unsigned)((rows + rows_per_block - 1) / rows_per_block));
    cfg.blockDim = dim3(256);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, split_merge_kernel, p, D);
}

template <int D>
static cudaError_t launch_tree_attention_t(const AttnMaps &m, const AttnParams &p, int num_sms,
                                           bool programmatic, cudaStream_t stream)
{
    static std::atomic<uint64_t> configured[2] = {{0}, {0}};
    if (p.split)
        return launch_attention_grid(tree_attention_kernel<D, true>, AttnLayout<D>::SMEM_BYTES, 352,
                                     configured[1], m, p, num_sms, programmatic, stream);
    return launch_attention_grid(tree_attention_kernel<D, false>, AttnLayout<D>::SMEM_BYTES, 352,
                                 configured[0], m, p, num_sms, programmatic, stream);
}

cudaError_t launch_tree_attention(const AttnMaps &m, const AttnParams &p, int D, int num_sms,
                                  bool programmatic, cudaStream_t stream)
{
    cudaError_t e;
    if (p.T_pad > 64) e = launch_tree_attention_rows(m, p, D, num_sms, programmatic, stream);
    else if (D == 128) e = launch_tree_attention_t<128>(m, p, num_sms, programmatic, stream);
    else e = launch_tree_attention_t<64>(m, p, num_sms, programmatic, stream);
    if (e != cudaSuccess || !p.split) return e;
    return launch_split_merge(p, D, attention_grid(p, num_sms), stream);
}

}  // namespace ppd
