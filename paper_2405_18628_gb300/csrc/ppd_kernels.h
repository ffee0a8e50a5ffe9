// ppd_kernels.h -- internal launch interface between the C-ABI layer
// (ppd_api.cu) and the kernels.  Not part of the public API.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace ppd {

// A bounded device-side wait gives up after this many nanoseconds of %globaltimer.
constexpr uint64_t kWaitLimitNs = 4000000000ull;

// Tensor maps of the attention operands (bf16, 128-byte swizzle, boxes of
// 64 columns): Q [LBH][T][D] (box rows T_pad), cache K/V [LBH][S_max][D] and
// tree K/V [LBH][T][D] (box rows 128).
struct AttnMaps {
    CUtensorMap q, kc, vc, kt, vt;
};

// The fused verification step's side work (see ppd_attention_common.cuh):
// argmax partials (from the preceding grid, or with in_grid computed by the
// side warps themselves), acceptance, and compaction of the CTA's own
// (layer, sequence, head) slices.
struct FusedStep {
    float *part_val;             // [B*T*splits] partial maxima
    int32_t *part_idx;
    int splits;
    // in_grid != 0: no preceding grid; the side warps compute the partial
    // maxima themselves while the other warps stream K/V.  Chunk c of the
    // [B*T][splits] partial grid is computed by CTA c mod grid; a CTA
    // publishes ready[cta] = tag once its chunks are written, where tag =
    // *epoch + 1 read at its start.  CTA 0 waits until every flag equals tag,
    // then sets *epoch = tag and *all_ready = tag; the other CTAs read
    // partials once *all_ready equals their tag.  Every call has a fresh tag,
    // so no flag needs zeroing.
    int in_grid;
    unsigned long long wait_limit_ns;   // the grid-wide wait gives up after this long
    int withhold_cta;            // diagnostics: this CTA never publishes its flag (-1: none)
    int chunk;                   // logits per chunk (multiple of 4 when vec)
    int vec;                     // 16-byte loads of the logits
    float stat_k;                // log2(e) / temperature (typical acceptance)
    unsigned long long *epoch;   // [1]
    unsigned long long *all_ready;   // [1]
    unsigned long long *ready;   // [grid]
    const int32_t *cand_tokens;  // [B,T]
    int32_t *argmax_out;         // [B,T]
    int32_t *accept_len;         // [B]
    int32_t *path;               // [B,T]
    int32_t *next_token;         // [B]
    int32_t *new_prefix_len;     // [B]
    int32_t *status;             // [B]: zeroed by the grid before (the argmax grid, or with
                                 // in_grid a one-block reset), then raised with atomicMax
    uint8_t *k_cache, *v_cache;  // raw cache storage
    const uint8_t *k_tree, *v_tree;
    int row_bytes;               // D * element size
    int V;
    int *scratch;                // [grid][kSideScratchInts] per-CTA scratch of the side warp
    // typical acceptance (typical != 0): partial softmax statistics from the
    // preceding grid, the logits for p(token), and the rule's parameters
    int typical;
    float *part_stats;           // [B*T*splits][3]
    const float *logits;         // [B,T,V]
    float inv_temp, epsilon, delta;
};

// Largest tree (nodes) of the verification step, and the per-warp scratch
// that acceptance needs: parents, then one 32-bit word per 32 nodes of pass bits.
constexpr int kMaxTree = 512;
constexpr int kAcceptScratchInts = kMaxTree + kMaxTree / 32;

// Per-CTA scratch of the fused step's side warp: acceptance scratch, top-1
// tokens, path, and (typical acceptance) each node's log-sum-exp and entropy.
constexpr int kSideScratchInts = kAcceptScratchInts + 4 * kMaxTree + 8;

struct AttnParams {
    const int32_t *prefix_len;  // [B]
    const int32_t *parent;      // [B,T]
    float *out;                 // [L,B,H,T,D]
    float *lse;                 // [L,B,H,T] or null
    int32_t *dev_status;        // [B] or null (main-loop errors; null in the fused step)
    int L, B, H, T, T_pad, S_max, n_units;
    int n_qb;                   // query blocks of 128 per (layer, sequence, head) slice
    int n_tt;                   // tree-key tiles of 128 per slice
    float scale_log2;           // softmax scale * log2(e)
    // Work split: split != 0 shares the units left after the full round-robin
    // rounds out by their key tiles (B <= kSplitMaxB); units cut by a range
    // boundary leave partial softmax states in split_part, merged afterwards by
    // launch_split_merge from the per-CTA records in split_rec.
    int split;
    float *split_part;          // [2 * grid][kSplitRows * (D + 2)] partial states
    struct SplitRecord *split_rec;   // [grid]
    int fused;                  // run the end phase below
    FusedStep fs;
    // Launched as a programmatic dependent of the preceding grid (a chain of
    // ppd_tree_attention calls): the setup that reads no input overlaps that
    // grid, then every thread waits for it before reading any input.
    int pdl_wait;
};

// Work split limits: batch size (the per-CTA range search holds the batch in
// two warp-wide registers), CTAs, and query rows of a partial state.
constexpr int kSplitMaxB = 64;
constexpr int kSplitMaxGrid = 256;
constexpr int kSplitRows = 128;

// The unit a CTA has to have merged: it holds the unit's first tile and its
// range ends inside the unit (u = -1: none).  off: the unit's tile 0 among
// the tail's tiles; n_tail: the tail's tile count.
struct SplitRecord {
    long long off, n_tail;
    int u, n_tiles;
};

// CTAs of an attention launch: one per SM, at most one per unit (with the
// work split: at most one per tile, and kSplitMaxGrid).
inline int attention_grid(const AttnParams &p, int num_sms)
{
    long long grid = num_sms;
    if (p.split) {
        const long long max_tiles = (long long)p.n_units * ((p.S_max + 127) / 128 + p.n_tt);
        grid = grid < kSplitMaxGrid ? grid : kSplitMaxGrid;
        grid = grid < max_tiles ? grid : max_tiles;
    } else {
        grid = grid < p.n_units ? grid : p.n_units;
    }
    return (int)grid;
}

// Merge the partial states of every cut unit of the attention launch just
// enqueued (one CTA per attention CTA, `grid` of them), after it completes.
cudaError_t launch_split_merge(const AttnParams &p, int D, int grid, cudaStream_t stream);

// Batches up to this size run the fused step (one grid, or an argmax grid then
// the attention grid).
constexpr int kFusedMaxB = 64;

// Dispatches on the padded tree size: up to 64 tokens the key-row kernel
// (ppd_attention.cu), 65..128 the query-row kernel (ppd_attention_rows.cu).
cudaError_t launch_tree_attention(const AttnMaps &m, const AttnParams &p, int D, int num_sms,
                                  bool programmatic, cudaStream_t stream);
cudaError_t launch_tree_attention_rows(const AttnMaps &m, const AttnParams &p, int D, int num_sms,
                                       bool programmatic, cudaStream_t stream);

// Splits per node row of the argmax: about 512 blocks over all rows, chunks of
// at least 2048 logits, at most 64 splits.
inline int argmax_split_count(int64_t rows, int V)
{
    if (rows <= 0) return 1;
    int64_t want = (512 + rows - 1) / rows;
    int64_t cap = V / 2048;
    if (cap > 64) cap = 64;
    if (cap < 1) cap = 1;
    if (want > cap) want = cap;
    if (want < 1) want = 1;
    return (int)want;
}

// Node argmax in two steps: per-(row, split) partial maxima, then a combine.
// part_stats (3 floats per partial) non-null: also the softmax statistics at
// `temperature` (typical acceptance).
cudaError_t launch_argmax_partials(const float *logits, int64_t rows, int V, int splits,
                                   float *part_val, int32_t *part_idx, float *part_stats,
                                   float temperature, int32_t *zero_status, int n_zero,
                                   cudaStream_t stream);
// The same partials from `grid` blocks of 512 threads (one warp per chunk at a
// time): the fused step's argmax grid on the SMs of its attention grid's last,
// partial round.
cudaError_t launch_argmax_narrow(const float *logits, int64_t rows, int V, int splits, int grid,
                                 float *part_val, int32_t *part_idx, float *part_stats,
                                 float temperature, int32_t *zero_status, int n_zero,
                                 cudaStream_t stream);
cudaError_t launch_argmax_combine(const float *part_val, const int32_t *part_idx, int64_t rows,
                                  int splits, int32_t *argmax_out, cudaStream_t stream);

struct AcceptArgs {
    const int32_t *cand_tokens;  // [B,T]
    const int32_t *parent;       // [B,T]
    const int32_t *prefix_len;   // [B]
    int32_t *accept_len;         // [B]
    int32_t *path;               // [B,T]
    int32_t *next_token;         // [B]
    int32_t *new_prefix_len;     // [B]
    int32_t *dev_status;         // [B]
    int T, V, S_max;
};

cudaError_t launch_accept_path(const int32_t *argmax, const AcceptArgs &a, int B,
                               cudaStream_t stream);

// argmax, natural-log log-sum-exp and entropy per row from stats partials.
cudaError_t launch_node_stats_combine(const float *part_val, const int32_t *part_idx,
                                      const float *part_stats, int64_t rows, int splits,
                                      int32_t *argmax_out, float *lse_out, float *ent_out,
                                      cudaStream_t stream);

cudaError_t launch_typical_accept(const float *logits, const float *lse, const float *ent,
                                  const int32_t *argmax, const AcceptArgs &a, int B,
                                  float temperature, float epsilon, float delta,
                                  cudaStream_t stream);

cudaError_t launch_kv_compact(void *k_cache, void *v_cache, const void *k_tree,
                              const void *v_tree, const int32_t *path,
                              const int32_t *accept_len, const int32_t *prefix_len, int L,
                              int B, int H, int T, int D, int S_max, int elem_bytes,
                              cudaStream_t stream);

// Next-step candidate tree: at most this many guesses per depth.
constexpr int kNextMaxK = 16;
constexpr int kNextMaxEpt = 128;
constexpr int kNextMaxSplit = 16;   // blocks sharing one row's columns

cudaError_t launch_next_tree(const float *logits, const int32_t *parent, const int32_t *cand,
                             const int32_t *path, const int32_t *accept_len,
                             const int32_t *next_token, int B, int T, int V, int n_states,
                             int T_next, const int32_t *tmpl_parent, const int32_t *tmpl_rank, int K,
                             int n_ept, int ept_mean, int32_t *topk, int32_t *kstate,
                             float *part_val, int32_t *part_idx, float *lse, int num_sms,
                             int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                             int32_t *status, cudaStream_t stream);

cudaError_t launch_round_bf16(const float *src, uint16_t *dst, int64_t n, cudaStream_t stream);

// Zero `n` status words once the preceding grid has completed, as a
// programmatic dependent launch that lets the next grid launch at once.
cudaError_t launch_zero_status(int32_t *status, int n, cudaStream_t stream);

cudaError_t launch_selftest_umma(const CUtensorMap &ma, const CUtensorMap &mb, const void *a_raw,
                                 const void *b_raw, float *d, int mode, int N, cudaStream_t stream);

}  // namespace ppd
