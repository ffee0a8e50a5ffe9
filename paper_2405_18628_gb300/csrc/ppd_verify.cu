// ppd_verify.cu -- node argmax, exact-matching acceptance, KV compaction,
// fp32 -> bf16 rounding, and the tensor-core layout self-test.
//
// Node argmax (paper Section 3 step (2): exact matching compares every guess
// token with the model's top-1 token at its parent) streams the fp32 logits
// with 16-byte loads, reduces (value, index) pairs with warp shuffles, and
// splits long rows over several blocks whose partial results are combined by
// the last block to finish.  Acceptance (Section 3 steps (2)-(3)) runs one
// warp per sequence: ballots build the bitset of matching nodes, each lane
// walks its nodes' root paths, and a warp max-reduction picks the deepest
// accepted node.  Compaction (Section 3 step (3)) copies the accepted rows
// into the cache with 16-byte loads and stores.
#include "ppd.h"
#include "ppd_accept.cuh"
#include "ppd_device.cuh"
#include "ppd_kernels.h"

#include <climits>
#include <cmath>
#include <mutex>

namespace ppd {

// ------------------------------------------------------------------ argmax

// Partial top-1 of rows of fp32 logits: block (row, s) scans columns
// [s*chunk, (s+1)*chunk) with 16-byte loads and writes its (value, index) to
// part_*[row * splits + s].  With kStats it also accumulates the softmax
// statistics (SoftStats, scale stat_k = log2(e) / temperature) of the same
// columns into part_stats[3 * (row * splits + s) ...] (m, s, t).  Block 0 also
// zeroes `zero_status` (the fused step's per-sequence status, raised later with
// atomicMax).  A grid launched after this one with programmatic stream
// serialization may start right away.
template <bool kVec, bool kStats>
__global__ void __launch_bounds__(256)
argmax_partial_kernel(const float *__restrict__ logits, int V, int splits, int chunk,
                      float *part_val, int32_t *part_idx, float *part_stats, float stat_k,
                      int32_t *zero_status, int n_zero)
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ float s_v[8];
    __shared__ int s_i[8];
    __shared__ float s_st[8][3];
    if (zero_status && blockIdx.x == 0)
        for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero_status[i] = 0;
    const int64_t row = blockIdx.x / splits;
    const int s = blockIdx.x % splits;
    const int lo = s * chunk;
    const int hi = min(V, lo + chunk);
    const float *x = logits + row * (int64_t)V;
    float bv = -INFINITY;
    int bi = INT_MAX;
    SoftStats st;
    auto take4 = [&](const float4 &f, int base) {
        consider(f.x, base, bv, bi);
        consider(f.y, base + 1, bv, bi);
        consider(f.z, base + 2, bv, bi);
        consider(f.w, base + 3, bv, bi);
        if (kStats) stats_add4(st, f.x * stat_k, f.y * stat_k, f.z * stat_k, f.w * stat_k);
    };
    if (kVec) {
        const float4 *x4 = reinterpret_cast<const float4 *>(x);
        const int n4_lo = lo >> 2, n4_hi = hi >> 2;
        int i = n4_lo + threadIdx.x;
        for (; i + 3 * 256 < n4_hi; i += 4 * 256) {
            float4 f[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) f[k] = __ldcs(x4 + i + k * 256);
#pragma unroll
            for (int k = 0; k < 4; ++k) take4(f[k], 4 * (i + k * 256));
        }
        for (; i < n4_hi; i += 256) take4(__ldcs(x4 + i), 4 * i);
    } else {
        // scalar loads; the statistics take one value at a time (three -inf pads)
        for (int i = lo + threadIdx.x; i < hi; i += 256) {
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
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        s_v[warp] = bv;
        s_i[warp] = bi;
        if (kStats) {
            s_st[warp][0] = st.m;
            s_st[warp][1] = st.s;
            s_st[warp][2] = st.t;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < 8; ++w) {
            consider(s_v[w], s_i[w], bv, bi);
            if (kStats) {
                SoftStats o;
                o.m = s_st[w][0];
                o.s = s_st[w][1];
                o.t = s_st[w][2];
                stats_merge(st, o);
            }
        }
        part_val[row * splits + s] = bv;
        part_idx[row * splits + s] = bi;
        if (kStats) {
            float *ps = part_stats + 3 * (row * splits + s);
            ps[0] = st.m;
            ps[1] = st.s;
            ps[2] = st.t;
        }
    }
}

__global__ void argmax_combine_kernel(const float *part_val, const int32_t *part_idx, int64_t rows,
                                      int splits, int32_t *argmax_out)
{
    const int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (row < rows) argmax_out[row] = combine_partials(part_val, part_idx, row, splits);
}

cudaError_t launch_argmax_partials(const float *logits, int64_t rows, int V, int splits,
                                   float *part_val, int32_t *part_idx, float *part_stats,
                                   float temperature, int32_t *zero_status, int n_zero,
                                   cudaStream_t stream)
{
    const bool vec = (V % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
    int chunk = (V + splits - 1) / splits;
    chunk = (chunk + 3) & ~3;
    const dim3 grid((unsigned)(rows * splits));
    const float k = part_stats ? 1.4426950408889634f / temperature : 0.f;
    if (part_stats) {
        if (vec)
            argmax_partial_kernel<true, true><<<grid, 256, 0, stream>>>(
                logits, V, splits, chunk, part_val, part_idx, part_stats, k, zero_status, n_zero);
        else
            argmax_partial_kernel<false, true><<<grid, 256, 0, stream>>>(
                logits, V, splits, chunk, part_val, part_idx, part_stats, k, zero_status, n_zero);
    } else {
        if (vec)
            argmax_partial_kernel<true, false><<<grid, 256, 0, stream>>>(
                logits, V, splits, chunk, part_val, part_idx, nullptr, 0.f, zero_status, n_zero);
        else
            argmax_partial_kernel<false, false><<<grid, 256, 0, stream>>>(
                logits, V, splits, chunk, part_val, part_idx, nullptr, 0.f, zero_status, n_zero);
    }
    return cudaGetLastError();
}

// The same partial maxima from a narrow grid: `gridDim.x` blocks of 512
// threads, each warp scanning (row, split) chunks c = warp, warp + all warps,
// ... with sixteen 16-byte loads per lane in flight.  The fused step launches
// it on as few SMs as hold the last, partial round of its attention grid, so
// the attention CTAs that must wait for those SMs are ones with a slice to
// spare.  Block 0 also zeroes `zero_status`; a grid launched after this one
// with programmatic stream serialization may start right away.
template <bool kStats>
__global__ void __launch_bounds__(512)
argmax_narrow_kernel(const float *__restrict__ logits, int V, int splits, int chunk, int vec,
                     int64_t n_chunks, float *part_val, int32_t *part_idx, float *part_stats,
                     float stat_k, int32_t *zero_status, int n_zero)
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (zero_status && blockIdx.x == 0)
        for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero_status[i] = 0;
    const int lane = threadIdx.x & 31;
    const int64_t n_warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t c = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); c < n_chunks;
         c += n_warps) {
        const int64_t row = c / splits;
        const int lo = (int)(c - row * splits) * chunk;
        const int hi = min(V, lo + chunk);
        float bv;
        int bi;
        SoftStats st;
        warp_logit_span<kStats, 16>(logits + row * (int64_t)V, lo, hi, vec != 0, stat_k, lane, bv, bi, st);
        if (lane == 0) {
            part_val[c] = bv;
            part_idx[c] = bi;
            if (kStats) {
                part_stats[3 * c] = st.m;
                part_stats[3 * c + 1] = st.s;
                part_stats[3 * c + 2] = st.t;
            }
        }
    }
}

cudaError_t launch_argmax_narrow(const float *logits, int64_t rows, int V, int splits, int grid,
                                 float *part_val, int32_t *part_idx, float *part_stats,
                                 float temperature, int32_t *zero_status, int n_zero,
                                 cudaStream_t stream)
{
    const int vec = (V % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
    const int chunk = (((V + splits - 1) / splits) + 3) & ~3;
    const int64_t n_chunks = rows * splits;
    if (part_stats)
        argmax_narrow_kernel<true><<<grid, 512, 0, stream>>>(logits, V, splits, chunk, vec, n_chunks,
                                                             part_val, part_idx, part_stats,
                                                             1.4426950408889634f / temperature,
                                                             zero_status, n_zero);
    else
        argmax_narrow_kernel<false><<<grid, 512, 0, stream>>>(logits, V, splits, chunk, vec, n_chunks,
                                                              part_val, part_idx, nullptr, 0.f,
                                                              zero_status, n_zero);
    return cudaGetLastError();
}

cudaError_t launch_argmax_combine(const float *part_val, const int32_t *part_idx, int64_t rows,
                                  int splits, int32_t *argmax_out, cudaStream_t stream)
{
    argmax_combine_kernel<<<(unsigned)((rows + 127) / 128), 128, 0, stream>>>(part_val, part_idx, rows,
                                                                              splits, argmax_out);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ accept

__global__ void __launch_bounds__(128)
accept_path_kernel(const int32_t *argmax, AcceptArgs a, int B)
{
    __shared__ int s_par[4][kAcceptScratchInts];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.x * 4 + warp;
    if (b >= B) return;
    const int32_t *top = argmax + (size_t)b * a.T;
    const AcceptResult r = accept_warp([&](int n) { return __ldg(top + n); }, a.parent + (size_t)b * a.T,
                                       a.cand_tokens + (size_t)b * a.T, __ldg(a.prefix_len + b), a.T,
                                       a.V, a.S_max, lane, s_par[warp], a.path + (size_t)b * a.T);
    if (lane == 0) {
        a.accept_len[b] = r.n_acc;
        a.next_token[b] = r.next_token;
        a.new_prefix_len[b] = r.new_prefix_len;
        a.dev_status[b] = r.status;
    }
}

cudaError_t launch_accept_path(const int32_t *argmax, const AcceptArgs &a, int B,
                               cudaStream_t stream)
{
    accept_path_kernel<<<(B + 3) / 4, 128, 0, stream>>>(argmax, a, B);
    return cudaGetLastError();
}

// Node statistics: argmax, natural-log log-sum-exp and entropy of each row
// from its partial results.
__global__ void node_stats_combine_kernel(const float *part_val, const int32_t *part_idx,
                                          const float *part_stats, int64_t rows, int splits,
                                          int32_t *argmax_out, float *lse_out, float *ent_out)
{
    const int64_t row = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (row >= rows) return;
    argmax_out[row] = combine_partials(part_val, part_idx, row, splits);
    const SoftStats st = combine_stats(part_stats, row, splits);
    stats_finish(st, lse_out[row], ent_out[row]);
}

cudaError_t launch_node_stats_combine(const float *part_val, const int32_t *part_idx,
                                      const float *part_stats, int64_t rows, int splits,
                                      int32_t *argmax_out, float *lse_out, float *ent_out,
                                      cudaStream_t stream)
{
    node_stats_combine_kernel<<<(unsigned)((rows + 127) / 128), 128, 0, stream>>>(
        part_val, part_idx, part_stats, rows, splits, argmax_out, lse_out, ent_out);
    return cudaGetLastError();
}

// Typical acceptance, one warp per sequence, from the node statistics.
__global__ void __launch_bounds__(128)
typical_accept_kernel(const float *logits, const float *lse, const float *ent,
                      const int32_t *argmax, AcceptArgs a, int B, float inv_temp, float epsilon,
                      float delta)
{
    __shared__ int s_par[4][kAcceptScratchInts];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.x * 4 + warp;
    if (b >= B) return;
    const size_t o = (size_t)b * a.T;
    const int32_t *top = argmax + o;
    const AcceptResult r = accept_warp_typical(
        [&](int n) { return __ldg(top + n); }, logits + o * a.V,
        [&](int n) { return __ldg(lse + o + n); }, [&](int n) { return __ldg(ent + o + n); },
        inv_temp, epsilon, delta, a.parent + o, a.cand_tokens + o, __ldg(a.prefix_len + b), a.T,
        a.V, a.S_max, lane, s_par[warp], a.path + o);
    if (lane == 0) {
        a.accept_len[b] = r.n_acc;
        a.next_token[b] = r.next_token;
        a.new_prefix_len[b] = r.new_prefix_len;
        a.dev_status[b] = r.status;
    }
}

cudaError_t launch_typical_accept(const float *logits, const float *lse, const float *ent,
                                  const int32_t *argmax, const AcceptArgs &a, int B,
                                  float temperature, float epsilon, float delta,
                                  cudaStream_t stream)
{
    typical_accept_kernel<<<(B + 3) / 4, 128, 0, stream>>>(logits, lse, ent, argmax, a, B,
                                                           1.0f / temperature, epsilon, delta);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ compaction

__global__ void __launch_bounds__(128)
kv_compact_kernel(uint8_t *kc, uint8_t *vc, const uint8_t *__restrict__ kt,
                  const uint8_t *__restrict__ vt, const int32_t *path, const int32_t *accept_len,
                  const int32_t *prefix_len, int64_t n_units, int B, int H, int T, int S_max,
                  int row_bytes)
{
    const int chunks = row_bytes >> 4;
    for (int64_t u = blockIdx.x; u < n_units; u += gridDim.x) {
        const int b = (int)((u / H) % B);
        const int n = __ldg(accept_len + b);
        const int P = __ldg(prefix_len + b);
        if (n <= 0 || n > T || P < 0 || (long long)P + n > S_max) continue;
        for (int w = threadIdx.x; w < n * chunks; w += blockDim.x) {
            const int j = w / chunks, c = w - j * chunks;
            const int src = __ldg(path + (size_t)b * T + j);
            if (src < 0 || src >= T) continue;
            const size_t so = ((size_t)u * T + src) * row_bytes + (size_t)c * 16;
            const size_t dof = ((size_t)u * S_max + P + j) * row_bytes + (size_t)c * 16;
            const uint4 kx = __ldg(reinterpret_cast<const uint4 *>(kt + so));
            const uint4 vx = __ldg(reinterpret_cast<const uint4 *>(vt + so));
            *reinterpret_cast<uint4 *>(kc + dof) = kx;
            *reinterpret_cast<uint4 *>(vc + dof) = vx;
        }
    }
}

cudaError_t launch_kv_compact(void *k_cache, void *v_cache, const void *k_tree,
                              const void *v_tree, const int32_t *path,
                              const int32_t *accept_len, const int32_t *prefix_len, int L,
                              int B, int H, int T, int D, int S_max, int elem_bytes,
                              cudaStream_t stream)
{
    const int64_t n_units = (int64_t)L * B * H;
    const int grid = (int)(n_units < 4096 ? n_units : 4096);
    kv_compact_kernel<<<grid, 128, 0, stream>>>(
        static_cast<uint8_t *>(k_cache), static_cast<uint8_t *>(v_cache),
        static_cast<const uint8_t *>(k_tree), static_cast<const uint8_t *>(v_tree), path,
        accept_len, prefix_len, n_units, B, H, T, S_max, D * elem_bytes);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ status reset

__global__ void zero_status_kernel(int32_t *status, int n)
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int i = threadIdx.x; i < n; i += blockDim.x) status[i] = 0;
}

cudaError_t launch_zero_status(int32_t *status, int n, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(128);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, zero_status_kernel, status, n);
}

// ------------------------------------------------------------------ fp32 -> bf16

__global__ void round_bf16_kernel(const float *__restrict__ src, uint16_t *__restrict__ dst,
                                  int64_t n)
{
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const __nv_bfloat16 h = __float2bfloat16_rn(src[i]);
        dst[i] = *reinterpret_cast<const uint16_t *>(&h);
    }
}

cudaError_t launch_round_bf16(const float *src, uint16_t *dst, int64_t n, cudaStream_t stream)
{
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 8192) blocks = 8192;
    round_bf16_kernel<<<(unsigned)blocks, 256, 0, stream>>>(src, dst, n);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ tensor-core self-test

constexpr uint32_t kSelfTestSmem = 200 * 1024;   // generous: operands use < 96 KB

__global__ void __launch_bounds__(128, 1)
selftest_umma_kernel(const __grid_constant__ CUtensorMap ma, const __grid_constant__ CUtensorMap mb,
                     const uint16_t *a_raw, const uint16_t *b_raw, float *d, int mode, int N)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    if (smem_addr(smem) & 1023u) return;
    uint8_t *sa = smem;                 // 32 KB
    uint8_t *sb = smem + 32 * 1024;     // up to 64 KB
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + 96 * 1024);   // [0] tma, [1] mma
    uint32_t *tmem_ptr = reinterpret_cast<uint32_t *>(smem + 96 * 1024 + 16);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + 96 * 1024 + 20);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        mbar_init(bar + 1, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 0) {
        tmem_alloc(tmem_ptr, 256);
        tmem_relinquish();
    }
    if (mode != 0) {
        // b given [128][N], N contiguous: thread t writes row t in the layout the
        // attention kernel uses for its probability tile.
        const int t = threadIdx.x;
        for (int n = 0; n < N; n += 8) {
            const uint4 v = *reinterpret_cast<const uint4 *>(b_raw + (size_t)t * N + n);
            const uint32_t addr = smem_addr(sb) + sw128_offset(t, n, 16384);
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x),
                         "r"(v.y), "r"(v.z), "r"(v.w)
                         : "memory");
        }
        fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_ptr;
    if (mode == 3) {
        // a given [128][256]: columns [0,128) the hi parts, [128,256) the lo parts of
        // a 128 x 128 A.  Thread t writes row t into TMEM columns 128.. in the layout
        // of the row-layout attention kernel's probability tile: per 32 keys, 16
        // columns of hi pairs followed by 16 columns of lo pairs.
        const int t = threadIdx.x;
        const uint32_t *row = reinterpret_cast<const uint32_t *>(a_raw + (size_t)t * 256);
        const uint32_t lane_off = (uint32_t)((t >> 5) * 32) << 16;
        for (int c = 0; c < 4; ++c) {
            uint32_t wh[16], wl[16];
            for (int i = 0; i < 16; ++i) {
                wh[i] = row[16 * c + i];
                wl[i] = row[64 + 16 * c + i];
            }
            tmem_st16(tmem + lane_off + 128 + 32 * c, wh);
            tmem_st16(tmem + lane_off + 128 + 32 * c + 16, wl);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }

    if (threadIdx.x == 0) {
        uint32_t tx = 0;
        if (mode == 0) tx = 128 * 128 * 2 + (uint32_t)N * 128 * 2;
        else if (mode != 3) tx = (mode == 1 ? 2u : 1u) * 16384u;
        mbar_arrive_expect_tx(bar, tx);
        if (mode == 0) {
            tma_load_2d(sa, &ma, bar, 0, 0);
            tma_load_2d(sa + 16384, &ma, bar, 64, 0);
            tma_load_2d(sb, &mb, bar, 0, 0);
            tma_load_2d(sb + (size_t)N * 128, &mb, bar, 64, 0);
        } else if (mode != 3) {
            tma_load_2d(sa, &ma, bar, 0, 0);
            if (mode == 1) tma_load_2d(sa + 16384, &ma, bar, 64, 0);
        }
        mbar_wait(bar, 0, abort_flag);
        tc_fence_after();
        if (!*abort_flag) {
            const uint32_t a0 = smem_addr(sa), b0 = smem_addr(sb);
            for (int kk = 0; kk < 8 && mode == 3; ++kk) {
                const uint32_t a_hi = tmem + 128 + 32 * (kk >> 1) + 8 * (kk & 1);
                const uint64_t db = make_smem_desc(b0 + kk * 2048, 16384, 1024);
                const uint32_t idesc = make_idesc_bf16(128, N, 0, 1);
                umma_bf16_ta(tmem, a_hi, db, idesc, kk > 0 ? 1u : 0u);
                umma_bf16_ta(tmem, a_hi + 16, db, idesc, 1u);
            }
            for (int kk = 0; kk < 8 && mode != 3; ++kk) {
                uint64_t da, db;
                uint32_t idesc;
                if (mode == 0) {
                    da = make_smem_desc(a0 + (kk >> 2) * 16384 + (kk & 3) * 32, 16, 1024);
                    db = make_smem_desc(b0 + (kk >> 2) * N * 128 + (kk & 3) * 32, 16, 1024);
                    idesc = make_idesc_bf16(128, N, 0, 0);
                } else {
                    da = make_smem_desc(a0 + kk * 2048, mode == 1 ? 16384u : 0u, 1024);
                    db = make_smem_desc(b0 + kk * 2048, 16384, 1024);
                    idesc = make_idesc_bf16(128, N, 1, 1);
                }
                umma_bf16(tmem, da, db, idesc, kk > 0 ? 1u : 0u);
            }
        }
        umma_commit(bar + 1);
    }
    __syncwarp();
    mbar_wait(bar + 1, 0, abort_flag);
    tc_fence_after();
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    for (int ch = 0; ch < N / 16; ++ch) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_off + ch * 16, r);
        tmem_wait_ld();
        for (int e = 0; e < 16; ++e)
            d[(size_t)(warp * 32 + lane) * N + ch * 16 + e] =
                *abort_flag ? NAN : __uint_as_float(r[e]);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 256);
}

cudaError_t launch_selftest_umma(const CUtensorMap &ma, const CUtensorMap &mb, const void *a_raw,
                                 const void *b_raw, float *d, int mode, int N, cudaStream_t stream)
{
    cudaError_t e = cudaFuncSetAttribute(selftest_umma_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSelfTestSmem);
    if (e != cudaSuccess) return e;
    selftest_umma_kernel<<<1, 128, kSelfTestSmem, stream>>>(
        ma, mb, static_cast<const uint16_t *>(a_raw), static_cast<const uint16_t *>(b_raw), d, mode,
        N);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ argmax without a workspace
//
// ppd_node_argmax_noalloc keeps its partial maxima in this fixed array instead of a
// caller-provided workspace.  Every GPU that loads the library holds it until the
// process exits.  Host code may not use the array's name as a device address: the
// address is looked up once per device with cudaGetSymbolAddress, with that device
// current, on the first call there.
namespace {

constexpr int64_t kNoAllocMaxPartials = 1 << 16;   // (row, split) pairs: 512 KiB in total

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocMaxPartials * 8];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mutex;
void *g_noalloc_addr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device (looked up once).
cudaError_t noalloc_scratch(void **addr)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (g_noalloc_addr[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_addr[dev] = p;
    }
    *addr = g_noalloc_addr[dev];
    return cudaSuccess;
}

}  // namespace

}  // namespace ppd

extern "C" ppd_status ppd_node_argmax_noalloc(const float *logits, int B, int T, int V,
                                              int32_t *argmax_out, void *stream)
{
    if (!logits || !argmax_out || B < 1 || T < 1 || V < 1) return PPD_ERR_INVALID_ARG;
    if ((double)B * T * V > 9.0e15) return PPD_ERR_INVALID_ARG;
    const int64_t rows = (int64_t)B * T;
    if (rows > ppd::kNoAllocMaxPartials) return PPD_ERR_UNSUPPORTED;   // B*T above the array's size
    int splits = ppd::argmax_split_count(rows, V);
    if (rows * splits > ppd::kNoAllocMaxPartials) splits = (int)(ppd::kNoAllocMaxPartials / rows);
    void *scratch = nullptr;
    if (ppd::noalloc_scratch(&scratch) != cudaSuccess) return PPD_ERR_CUDA;
    float *pv = static_cast<float *>(scratch);
    int32_t *pi = reinterpret_cast<int32_t *>(static_cast<unsigned char *>(scratch) +
                                              ppd::kNoAllocMaxPartials * 4);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (ppd::launch_argmax_partials(logits, rows, V, splits, pv, pi, nullptr, 1.f, nullptr, 0, s) !=
        cudaSuccess)
        return PPD_ERR_CUDA;
    return ppd::launch_argmax_combine(pv, pi, rows, splits, argmax_out, s) == cudaSuccess ? PPD_OK
                                                                                          : PPD_ERR_CUDA;
}

