// ppd_kernels.h -- internal launch interface between the C-ABI layer
// (ppd_api.cu) and the kernels.  Not part of the public API.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace ppd {

// Tensor maps of the attention operands (bf16, 128-byte swizzle, boxes of
// 64 columns): Q [LBH][T][D] (box rows T_pad), cache K/V [LBH][S_max][D] and
// tree K/V [LBH][T][D] (box rows 128).
struct AttnMaps {
    CUtensorMap q, kc, vc, kt, vt;
};

struct AttnParams {
    const int32_t *prefix_len;  // [B]
    const int32_t *parent;      // [B,T]
    float *out;                 // [L,B,H,T,D]
    float *lse;                 // [L,B,H,T] or null
    int32_t *dev_status;        // [B] or null
    int L, B, H, T, T_pad, S_max, n_units;
    float scale_log2;           // softmax scale * log2(e)
};

cudaError_t launch_tree_attention(const AttnMaps &m, const AttnParams &p, int D, int num_sms,
                                  cudaStream_t stream);

// Node argmax over rows of fp32 logits, split over `splits` blocks per row
// with a last-block combine.  When `acc` is non-null, the block that
// finishes the last row of a sequence also runs the acceptance rule for it.
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

struct ArgmaxScratch {
    float *part_val;       // [rows * splits]
    int32_t *part_idx;     // [rows * splits]
    int32_t *row_count;    // [rows]   zero on entry, left zero on exit
    int32_t *seq_count;    // [B]      zero on entry, left zero on exit
};

cudaError_t launch_node_argmax(const float *logits, int64_t rows, int V, int splits,
                               int32_t *argmax_out, const ArgmaxScratch &ws,
                               const AcceptArgs *acc, int B, cudaStream_t stream);

cudaError_t launch_accept_path(const int32_t *argmax, const AcceptArgs &a, int B,
                               cudaStream_t stream);

cudaError_t launch_kv_compact(void *k_cache, void *v_cache, const void *k_tree,
                              const void *v_tree, const int32_t *path,
                              const int32_t *accept_len, const int32_t *prefix_len, int L,
                              int B, int H, int T, int D, int S_max, int elem_bytes,
                              cudaStream_t stream);

cudaError_t launch_round_bf16(const float *src, uint16_t *dst, int64_t n, cudaStream_t stream);

cudaError_t launch_selftest_umma(const CUtensorMap &ma, const CUtensorMap &mb, const void *b_raw,
                                 float *d, int mode, int N, cudaStream_t stream);

}  // namespace ppd
