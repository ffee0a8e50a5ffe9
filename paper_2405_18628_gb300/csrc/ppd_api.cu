// ppd_api.cu -- the C ABI of libppd (declared in include/ppd.h): host-side
// argument checks, workspace layout, TMA tensor-map encoding and the launch
// sequence of each entry point.  No entry point allocates, frees or
// synchronises; all work is enqueued on the caller's stream.
#include "ppd.h"
#include "ppd_kernels.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <atomic>
#include <cstring>
#include <mutex>

namespace {

using ppd::AcceptArgs;
using ppd::AttnMaps;
using ppd::AttnParams;

constexpr int kMaxT = ppd::kMaxTree;   // tree tokens per sequence
constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// byte ranges [a, a+na) and [b, b+nb) intersect
bool overlaps(const void *a, size_t na, const void *b, size_t nb)
{
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + nb && y < x + na;
}

int num_sms()
{
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cache[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        cache[dev] = n;
    }
    return cache[dev];
}

int argmax_splits(int64_t rows, int V) { return ppd::argmax_split_count(rows, V); }

// Workspace: the in-grid argmax's sync words, the argmax partials, the side
// warp's scratch, the bf16 copies of fp32 operands, then the work split's
// per-CTA records and partial states.
struct WsLayout {
    size_t part_val, part_idx, part_stats, node_lse, node_ent, side, sync, conv, split_rec,
        split_part, total;
    int splits;
};

int split_grid() { return num_sms() < ppd::kSplitMaxGrid ? num_sms() : ppd::kSplitMaxGrid; }

// Logits per (row, split) chunk of the argmax (a multiple of 4), and whether
// the rows can be read with 16-byte loads; as launch_argmax_partials does.
int argmax_chunk(int V, int splits) { return (((V + splits - 1) / splits) + 3) & ~3; }
int argmax_vec(const float *logits, int V)
{
    return (V % 4 == 0) && ((reinterpret_cast<uintptr_t>(logits) & 15) == 0);
}

// The fused step computes the node argmax inside the attention grid (one
// side warp per CTA, while the other warps stream K/V) when the logits are a
// small share of the bytes the attention streams.  A side warp keeps 2 KB in
// flight (deeper bursts slow the attention more than they gain) and, with the
// HBM saturated by the K/V stream, reads about 1 GB/s against its CTA's
// ~42 GB/s of K/V.  Measured at Vicuna-7B shapes with a growing vocabulary:
// in-grid beats the two-grid form while the logits are at most 1/70 of the
// K/V bytes, and the side warps become the bottleneck at 1/35.  Otherwise a
// separate argmax grid runs first.  S_max bounds the prefix lengths, which
// only the device knows.
#ifndef PPD_IN_GRID_MIN_RATIO
#define PPD_IN_GRID_MIN_RATIO 64
#endif
bool in_grid_argmax_pays(int L, int B, int H, int T, int D, int V, int S_max)
{
    const double kv = 4.0 * L * B * H * ((double)S_max + T) * D;
    const double logits = 4.0 * B * (double)T * V;
    return logits * PPD_IN_GRID_MIN_RATIO <= kv;
}

// Forms of the fused step (ppd_verify_step_form): separate grids for large
// batches; an argmax grid then the attention grid; one grid whose side warps
// compute the argmax partials while the K/V stream runs.
enum FusedForm { kFormGrids = 0, kFormTwoGrids = 1, kFormSide = 2 };

// A form forced by ppd_set_verify_step_form (-1: chosen by the rules below).
std::atomic<int> g_forced_form{-1};

// The in-grid argmax's grid-wide wait: its limit in ns (0: the default of the
// device-side waits) and a CTA that withholds its flag (-1: none); set only by
// ppd_debug_grid_wait, for tests of the timeout path.
std::atomic<unsigned long long> g_grid_wait_ns{0};
std::atomic<int> g_withhold_cta{-1};

int narrow_argmax_grid(int L, int B, int H, int T, int D, int V, int S_max);

// The form of a fused step (B <= kFusedMaxB) of these sizes: an argmax grid
// first when it fits on the idle SMs of the attention grid's last, partial
// round (measured at Vicuna-7B shapes: 181.9 us against 183.2 us with the
// side warps; equal at Vicuna-13B and on the batch-8 sweep), else the side
// warps when the logits are a small enough share of the K/V bytes, else an
// argmax grid over every SM.
int choose_form(int L, int B, int H, int T, int D, int V, int S_max)
{
    const int forced = g_forced_form.load(std::memory_order_relaxed);
    if (forced >= kFormTwoGrids) return forced;
    if (narrow_argmax_grid(L, B, H, T, D, V, S_max) > 0) return kFormTwoGrids;
    return in_grid_argmax_pays(L, B, H, T, D, V, S_max) ? kFormSide : kFormTwoGrids;
}

WsLayout workspace_layout(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt)
{
    WsLayout w{};
    const int64_t rows = (int64_t)B * T;
    w.splits = argmax_splits(rows, V);
    size_t off = 0;
    // the in-grid argmax's epoch and all-ready words and per-CTA flags first, at
    // the same offset for every size: a workspace reused for another shape
    // keeps them in place, so its flags only ever hold tags of earlier calls
    w.sync = off;
    off = align_up(off + (size_t)(2 + ppd::kSplitMaxGrid) * 8);
    const size_t cap = (size_t)rows * (size_t)w.splits;
    w.part_val = off;
    off = align_up(off + cap * 4);
    w.part_idx = off;
    off = align_up(off + cap * 4);
    w.part_stats = off;   // softmax statistics partials (typical acceptance)
    off = align_up(off + cap * 12);
    w.node_lse = off;
    off = align_up(off + (size_t)rows * 4);
    w.node_ent = off;
    off = align_up(off + (size_t)rows * 4);
    w.side = off;
    off = align_up(off + (size_t)num_sms() * ppd::kSideScratchInts * 4);
    w.conv = off;
    if (dt == PPD_F32) {
        const size_t lbh = (size_t)L * B * H;
        off = align_up(off + lbh * ((size_t)3 * T + 2 * (size_t)S_max) * D * 2);
    }
    w.split_rec = off;
    off = align_up(off + (size_t)split_grid() * sizeof(ppd::SplitRecord));
    w.split_part = off;
    off = align_up(off + (size_t)2 * split_grid() * ppd::kSplitRows * (D + 2) * sizeof(float));
    w.total = off;
    return w;
}

// ------------------------------------------------------------------ tensor maps

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// bf16 tensor viewed as [depth][rows][inner], box {64, box_rows, 1}, 128-byte swizzle,
// out-of-range rows read as zero.
bool encode_3d(CUtensorMap *m, const void *base, uint64_t inner, uint64_t rows, uint64_t depth,
               uint32_t box_rows)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[3] = {inner, rows, depth};
    const cuuint64_t strides[2] = {inner * 2, inner * 2 * rows};
    const cuuint32_t box[3] = {64, box_rows, 1};
    const cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_2d(CUtensorMap *m, const void *base, uint64_t inner, uint64_t rows, uint32_t box_rows)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {inner, rows};
    const cuuint64_t strides[1] = {inner * 2};
    const cuuint32_t box[2] = {64, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The CUDA error behind the latest PPD_ERR_CUDA of this process (diagnostics).
std::atomic<int> g_last_cuda_error{cudaSuccess};

// A launch reported failed through the runtime's last error (kernels launched
// with <<< >>>): record it and clear it.
ppd_status cuda_failed()
{
    const cudaError_t e = cudaGetLastError();
    g_last_cuda_error.store((int)(e != cudaSuccess ? e : cudaErrorUnknown), std::memory_order_relaxed);
    return PPD_ERR_CUDA;
}

// A failed call clears the runtime's last-error state (errors that do not
// break the context), so it cannot surface as the status of a later call.
ppd_status cuda_status(cudaError_t e)
{
    if (e == cudaSuccess) return PPD_OK;
    g_last_cuda_error.store((int)e, std::memory_order_relaxed);
    (void)cudaGetLastError();
    return PPD_ERR_CUDA;
}

// ------------------------------------------------------------------ shared checks

bool attn_dims_ok(int L, int B, int H, int T, int D, int S_max, ppd_dtype dt)
{
    if (L < 1 || B < 1 || H < 1 || T < 1 || T > kMaxT || S_max < 1) return false;
    if (D != 64 && D != 128) return false;
    if (dt != PPD_BF16 && dt != PPD_F32) return false;
    const double lbh = (double)L * B * H;
    if (lbh > 2147483647.0 || lbh * S_max * D > 9.0e15) return false;
    return true;
}

// Enqueue the attention of all L*B*H slices (bf16 operands).
// Does sharing the launch's key tiles over all SMs (the work split) beat one
// whole slice per SM?  Only launches with fewer slices than SMs can gain (with
// more, the last round's idle SMs cost less than the merge; measured on the
// Vicuna-7B/13B and MobileLlama shapes).  Counted in tiles of 128 keys, with
// S_max standing in for the (device-side) prefix lengths: one round of whole
// slices takes t_u tiles; the split takes its share of all tiles plus about
// kSplitCostTiles for the range planning and the merge grid.
constexpr long long kSplitCostTiles = 6;

bool split_pays(const AttnParams &p, int sms)
{
    if (p.n_units >= sms) return false;
    const long long t_u = (p.S_max + 127) / 128 + p.n_tt;
    const long long share = ((long long)p.n_units * t_u + sms - 1) / sms;
    return share + kSplitCostTiles < t_u;
}

// Whether an attention launch of these sizes, given a workspace, shares its key
// tiles out (the work split): a batch of at most kSplitMaxB and a launch that
// gains from it.
bool attention_splits(int L, int B, int H, int T, int S_max)
{
    if (B > ppd::kSplitMaxB) return false;
    AttnParams p{};
    const int T_pad = (T + 31) & ~31;
    p.S_max = S_max;
    p.n_qb = T_pad > 64 ? (T + 127) / 128 : 1;
    p.n_tt = p.n_qb;
    p.n_units = (int)((long long)L * B * H) * p.n_qb;
    return split_pays(p, split_grid());
}

// With a workspace of the full layout and attention_splits(...), the key tiles
// are shared evenly over the CTAs (see ppd_attention_common.cuh).
ppd_status enqueue_attention(const void *q, const void *kc, const void *vc, const void *kt,
                             const void *vt, const int32_t *prefix_len, const int32_t *parent,
                             int L, int B, int H, int T, int D, int S_max, float scale, float *out,
                             float *lse, int32_t *dev_status, uint8_t *ws, const WsLayout *wl,
                             const ppd::FusedStep *fused, bool programmatic, bool chained,
                             cudaStream_t stream)
{
    const int T_pad = (T + 31) & ~31;
    const uint64_t lbh = (uint64_t)L * B * H;
    // trees of more than 64 tokens run the row-layout kernel, which reads Q in
    // boxes of 128 rows (rows past T arrive as zeros)
    const uint32_t q_box = T_pad > 64 ? 128u : (uint32_t)T_pad;
    AttnMaps m;
    if (!encode_3d(&m.q, q, D, T, lbh, q_box) || !encode_3d(&m.kc, kc, D, S_max, lbh, 128) ||
        !encode_3d(&m.vc, vc, D, S_max, lbh, 128) || !encode_3d(&m.kt, kt, D, T, lbh, 128) ||
        !encode_3d(&m.vt, vt, D, T, lbh, 128))
        return PPD_ERR_CUDA;
    AttnParams p{};
    p.prefix_len = prefix_len;
    p.parent = parent;
    p.out = out;
    p.lse = lse;
    p.dev_status = dev_status;
    p.L = L;
    p.B = B;
    p.H = H;
    p.T = T;
    p.T_pad = T_pad;
    p.S_max = S_max;
    // trees of more than 64 tokens: slices split into blocks of 128 query rows,
    // the tree keys into tiles of 128
    p.n_qb = T_pad > 64 ? (T + 127) / 128 : 1;
    p.n_tt = T_pad > 64 ? (T + 127) / 128 : 1;
    p.n_units = (int)lbh * p.n_qb;
    const float sc = scale > 0.f ? scale : 1.0f / std::sqrt((float)D);
    p.scale_log2 = sc * 1.4426950408889634f;
    if (ws && wl && attention_splits(L, B, H, T, S_max)) {
        p.split = 1;
        p.split_rec = reinterpret_cast<ppd::SplitRecord *>(ws + wl->split_rec);
        p.split_part = reinterpret_cast<float *>(ws + wl->split_part);
    }
    p.fused = fused != nullptr;
    if (fused) p.fs = *fused;
    p.pdl_wait = chained ? 1 : 0;
    return cuda_status(ppd::launch_tree_attention(m, p, D, split_grid(), programmatic || chained,
                                                  stream));
}

// fp32 operands: round to bf16 copies in the workspace first.
ppd_status enqueue_attention_any(const void *q, const void *kc, const void *vc, const void *kt,
                                 const void *vt, const int32_t *prefix_len, const int32_t *parent,
                                 int L, int B, int H, int T, int D, int S_max, ppd_dtype dt,
                                 float scale, float *out, float *lse, int32_t *dev_status,
                                 uint8_t *ws, const WsLayout &wl, const ppd::FusedStep *fused,
                                 cudaStream_t stream, bool chained = false)
{
    // With bf16 operands the attention grid only reads caller inputs before its end
    // phase, so it may overlap the preceding (argmax) grid -- when there is one.
    // `chained`: the grid follows a status reset launched as a programmatic
    // dependent, and waits for it (and so for whatever preceded it) itself.
    if (dt == PPD_BF16)
        return enqueue_attention(q, kc, vc, kt, vt, prefix_len, parent, L, B, H, T, D, S_max, scale,
                                 out, lse, dev_status, ws, ws ? &wl : nullptr, fused,
                                 fused != nullptr && !fused->in_grid, chained, stream);
    const int64_t lbh = (int64_t)L * B * H;
    const int64_t n_t = lbh * T * D, n_c = lbh * (int64_t)S_max * D;
    uint16_t *bq = reinterpret_cast<uint16_t *>(ws + wl.conv);
    uint16_t *bkt = bq + n_t;
    uint16_t *bvt = bkt + n_t;
    uint16_t *bkc = bvt + n_t;
    uint16_t *bvc = bkc + n_c;
    if (ppd::launch_round_bf16((const float *)q, bq, n_t, stream) != cudaSuccess ||
        ppd::launch_round_bf16((const float *)kt, bkt, n_t, stream) != cudaSuccess ||
        ppd::launch_round_bf16((const float *)vt, bvt, n_t, stream) != cudaSuccess ||
        ppd::launch_round_bf16((const float *)kc, bkc, n_c, stream) != cudaSuccess ||
        ppd::launch_round_bf16((const float *)vc, bvc, n_c, stream) != cudaSuccess)
        return cuda_failed();
    return enqueue_attention(bq, bkc, bvc, bkt, bvt, prefix_len, parent, L, B, H, T, D, S_max,
                             scale, out, lse, dev_status, ws, &wl, fused, false, false, stream);
}

// Blocks of the fused step's narrow argmax grid (0: use the wide grid).  When
// the attention grid's slices do not fill whole rounds, the CTAs of the last,
// partial round that hold one slice fewer -- grid - (n_units mod grid) of
// them -- have a slice's time to spare; the argmax blocks take as many SMs
// (at most half of them), the CTAs dispatched last, which are those, wait for
// them, and nothing on the critical path does.  Each block's share of the
// logits must then be at most half a slice's K/V bytes (S_max standing in for
// the device-side prefix lengths).  The work split (fewer slices than SMs)
// leaves no CTA with time to spare.
int narrow_argmax_grid(int L, int B, int H, int T, int D, int V, int S_max)
{
    if (attention_splits(L, B, H, T, S_max)) return 0;
    const int T_pad = (T + 31) & ~31;
    const long long n_qb = T_pad > 64 ? (T + 127) / 128 : 1;
    const long long n_units = (long long)L * B * H * n_qb;
    const long long grid = n_units < split_grid() ? n_units : split_grid();
    const long long r = n_units % grid;
    if (r == 0) return 0;
    long long g = grid - r;
    if (g > num_sms() / 2) g = num_sms() / 2;
    if (g < 8) return 0;
    const double logits = 4.0 * B * (double)T * V;
    const double slice = 4.0 * ((double)S_max + T) * D;
    return logits / (double)g <= slice / 2 ? (int)g : 0;
}

}  // namespace

// Parameters of typical acceptance (null: exact matching).
struct TypicalParams {
    float temperature, epsilon, delta;
};

static ppd_status verify_step_impl(const void *q, void *k_cache, void *v_cache,
                                   const void *k_tree, const void *v_tree,
                                   const int32_t *prefix_len, const int32_t *parent,
                                   const int32_t *cand_tokens, const float *logits, int L, int B,
                                   int H, int T, int D, int V, int S_max, ppd_dtype dt, float scale,
                                   const TypicalParams *typ, float *out, float *lse,
                                   int32_t *argmax_out, int32_t *accept_len, int32_t *path,
                                   int32_t *next_token, int32_t *new_prefix_len,
                                   int32_t *dev_status, void *workspace, size_t ws_bytes,
                                   void *stream)
{
    if (!q || !k_cache || !v_cache || !k_tree || !v_tree || !prefix_len || !parent ||
        !cand_tokens || !logits || !out || !argmax_out || !accept_len || !path || !next_token ||
        !new_prefix_len || !dev_status || !workspace)
        return PPD_ERR_INVALID_ARG;
    if (!attn_dims_ok(L, B, H, T, D, S_max, dt) || V < 1 || !std::isfinite(scale))
        return PPD_ERR_INVALID_ARG;
    if ((double)B * T * V > 9.0e15) return PPD_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(k_tree, 16) ||
        !aligned(v_tree, 16) || !aligned(out, 4) || !aligned(lse, 4))
        return PPD_ERR_INVALID_ARG;
    const int eb = dt == PPD_BF16 ? 2 : 4;
    const size_t lbh = (size_t)L * B * H;
    const size_t nc = lbh * S_max * D * eb, nt = lbh * T * D * eb;
    if (overlaps(k_cache, nc, k_tree, nt) || overlaps(k_cache, nc, v_tree, nt) ||
        overlaps(v_cache, nc, k_tree, nt) || overlaps(v_cache, nc, v_tree, nt) ||
        overlaps(k_cache, nc, v_cache, nc))
        return PPD_ERR_INVALID_ARG;
    const WsLayout wl = workspace_layout(L, B, H, T, D, V, S_max, dt);
    if (ws_bytes < wl.total || !aligned(workspace, kAlign)) return PPD_ERR_INVALID_ARG;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float *pv = reinterpret_cast<float *>(ws + wl.part_val);
    int32_t *pi = reinterpret_cast<int32_t *>(ws + wl.part_idx);
    float *pst = typ ? reinterpret_cast<float *>(ws + wl.part_stats) : nullptr;
    const float temp = typ ? typ->temperature : 1.f;
    const int64_t rows = (int64_t)B * T;

    if (B <= ppd::kFusedMaxB) {
        bool in_grid = choose_form(L, B, H, T, D, V, S_max) == kFormSide;
        while (true) {
            // 1. partial maxima (and statistics) of every node's logits; also zeroes
            //    dev_status.  In-grid: the attention grid's side warps do this instead.
            if (!in_grid) {
                const int narrow = narrow_argmax_grid(L, B, H, T, D, V, S_max);
                const cudaError_t e =
                    narrow > 0 ? ppd::launch_argmax_narrow(logits, rows, V, wl.splits, narrow, pv, pi, pst,
                                                           temp, dev_status, B, s)
                               : ppd::launch_argmax_partials(logits, rows, V, wl.splits, pv, pi, pst, temp,
                                                             dev_status, B, s);
                if (e != cudaSuccess) return cuda_status(e);
            }
            // 2. attention over every layer, overlapping step 1; its side warps combine
            //    the argmax, decide acceptance and compact the accepted rows
            ppd::FusedStep f{};
            f.part_val = pv;
            f.part_idx = pi;
            f.splits = wl.splits;
            f.cand_tokens = cand_tokens;
            f.argmax_out = argmax_out;
            f.accept_len = accept_len;
            f.path = path;
            f.next_token = next_token;
            f.new_prefix_len = new_prefix_len;
            f.status = dev_status;
            f.k_cache = static_cast<uint8_t *>(k_cache);
            f.v_cache = static_cast<uint8_t *>(v_cache);
            f.k_tree = static_cast<const uint8_t *>(k_tree);
            f.v_tree = static_cast<const uint8_t *>(v_tree);
            f.row_bytes = D * eb;
            f.V = V;
            f.scratch = reinterpret_cast<int *>(ws + wl.side);
            f.logits = logits;
            if (in_grid) {
                f.in_grid = 1;
                f.chunk = argmax_chunk(V, wl.splits);
            }
            if (in_grid) {
                // no argmax grid to zero the status first: a one-block reset does,
                // so that every status write can be an atomic maximum
                if (ppd::launch_zero_status(dev_status, B, s) != cudaSuccess) return cuda_failed();
                const unsigned long long lim = g_grid_wait_ns.load(std::memory_order_relaxed);
                f.wait_limit_ns = lim ? lim : ppd::kWaitLimitNs;
                f.withhold_cta = g_withhold_cta.load(std::memory_order_relaxed);
                f.vec = argmax_vec(logits, V);
                f.stat_k = 1.4426950408889634f / temp;
                f.epoch = reinterpret_cast<unsigned long long *>(ws + wl.sync);
                f.all_ready = f.epoch + 1;
                f.ready = f.epoch + 2;
            }
            if (typ) {
                f.typical = 1;
                f.part_stats = pst;
                f.inv_temp = 1.f / typ->temperature;
                f.epsilon = typ->epsilon;
                f.delta = typ->delta;
            }
            const ppd_status st = enqueue_attention_any(q, k_cache, v_cache, k_tree, v_tree,
                                                        prefix_len, parent, L, B, H, T, D, S_max,
                                                        dt, scale, out, lse, nullptr, ws, wl, &f, s);
            if (st == PPD_OK || !in_grid) return st;
            // the cooperative launch could not have every CTA resident (SMs taken by
            // other work): clear its error and run the argmax as its own grid
            if (g_last_cuda_error.load(std::memory_order_relaxed) != cudaErrorCooperativeLaunchTooLarge)
                return st;
            in_grid = false;
        }
    }

    // large batches: the same steps as separate grids
    AcceptArgs a{cand_tokens, parent, prefix_len, accept_len, path, next_token, new_prefix_len,
                 dev_status, T, V, S_max};
    if (ppd::launch_argmax_partials(logits, rows, V, wl.splits, pv, pi, pst, temp, nullptr, 0, s) !=
        cudaSuccess)
        return cuda_failed();
    if (typ) {
        float *nl = reinterpret_cast<float *>(ws + wl.node_lse);
        float *ne = reinterpret_cast<float *>(ws + wl.node_ent);
        if (ppd::launch_node_stats_combine(pv, pi, pst, rows, wl.splits, argmax_out, nl, ne, s) !=
                cudaSuccess ||
            ppd::launch_typical_accept(logits, nl, ne, argmax_out, a, B, typ->temperature,
                                       typ->epsilon, typ->delta, s) != cudaSuccess)
            return cuda_failed();
    } else {
        if (ppd::launch_argmax_combine(pv, pi, rows, wl.splits, argmax_out, s) != cudaSuccess ||
            ppd::launch_accept_path(argmax_out, a, B, s) != cudaSuccess)
            return cuda_failed();
    }
    ppd_status st = enqueue_attention_any(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent,
                                          L, B, H, T, D, S_max, dt, scale, out, lse, dev_status,
                                          ws, wl, nullptr, s);
    if (st != PPD_OK) return st;
    return cuda_status(ppd::launch_kv_compact(k_cache, v_cache, k_tree, v_tree, path, accept_len,
                                              prefix_len, L, B, H, T, D, S_max, eb, s));
}

int ppd_verify_step_form(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt)
{
    if (!attn_dims_ok(L, B, H, T, D, S_max, dt) || V < 1) return -1;
    if (B > ppd::kFusedMaxB) return kFormGrids;
    return choose_form(L, B, H, T, D, V, S_max);
}

ppd_status ppd_debug_grid_wait(unsigned long long limit_ns, int withhold_cta)
{
    if (withhold_cta < -1) return PPD_ERR_INVALID_ARG;
    g_grid_wait_ns.store(limit_ns);
    g_withhold_cta.store(withhold_cta);
    return PPD_OK;
}

int ppd_set_verify_step_form(int form)
{
    if (form != -1 && form != kFormTwoGrids && form != kFormSide) return -2;
    return g_forced_form.exchange(form);
}

int ppd_verify_step_launches(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt,
                             int typical)
{
    (void)typical;   // both acceptance rules launch the same number of kernels
    const int form = ppd_verify_step_form(L, B, H, T, D, V, S_max, dt);
    if (form < 0) return -1;
    const int round = dt == PPD_F32 ? 5 : 0;   // fp32 -> bf16 copies of Q, K/V tree, K/V cache
    const int attn = attention_splits(L, B, H, T, S_max) ? 2 : 1;   // + the merge grid
    if (form == kFormTwoGrids) return 1 + round + attn;
    if (form == kFormSide) return 1 + round + attn;   // the status reset, then one grid
    // partial maxima, combine (or statistics), acceptance, attention, compaction
    return 3 + round + attn + 1;
}

static bool typical_params_ok(float temperature, float epsilon, float delta)
{
    return std::isfinite(temperature) && temperature > 0.f && std::isfinite(epsilon) &&
           std::isfinite(delta) && std::isfinite(1.f / temperature);
}

extern "C" {

size_t ppd_workspace_bytes(int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt)
{
    if (L < 1 || B < 1 || H < 1 || T < 1 || D < 1 || V < 1 || S_max < 0) return 0;
    return workspace_layout(L, B, H, T, D, V, S_max, dt).total;
}


const char *ppd_last_cuda_error(void)
{
    return cudaGetErrorName((cudaError_t)g_last_cuda_error.load(std::memory_order_relaxed));
}

const char *ppd_status_string(ppd_status s)
{
    switch (s) {
    case PPD_OK: return "ok";
    case PPD_ERR_INVALID_ARG: return "invalid argument";
    case PPD_ERR_UNSUPPORTED: return "unsupported configuration";
    case PPD_ERR_TREE: return "malformed tree or token id";
    case PPD_ERR_CAPACITY: return "cache capacity exceeded or prefix length out of range";
    case PPD_ERR_CUDA: return "CUDA runtime error";
    case PPD_ERR_TIMEOUT: return "device-side wait timed out";
    }
    return "unknown status";
}

ppd_status ppd_tree_attention(const void *q, const void *k_cache, const void *v_cache,
                              const void *k_tree, const void *v_tree,
                              const int32_t *prefix_len, const int32_t *parent,
                              int L, int B, int H, int T, int D, int S_max, ppd_dtype dt,
                              float scale, float *out, float *lse, int32_t *dev_status,
                              void *workspace, size_t ws_bytes, void *stream)
{
    if (!q || !k_cache || !v_cache || !k_tree || !v_tree || !prefix_len || !parent || !out ||
        !dev_status)
        return PPD_ERR_INVALID_ARG;
    if (!attn_dims_ok(L, B, H, T, D, S_max, dt) || !std::isfinite(scale)) return PPD_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(k_tree, 16) ||
        !aligned(v_tree, 16) || !aligned(out, 4) || !aligned(lse, 4))
        return PPD_ERR_INVALID_ARG;
    const WsLayout wl = workspace_layout(L, B, H, T, D, 1, S_max, dt);
    const bool ws_ok = workspace && ws_bytes >= wl.total && aligned(workspace, kAlign);
    if (dt == PPD_F32 && !ws_ok) return PPD_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // dev_status is reset by a one-block grid launched as a programmatic
    // dependent (it waits for the preceding grid before writing); the attention
    // grid is its programmatic dependent in turn, so a sequence of calls (one
    // per layer, as a model runs them) launches each grid while the previous
    // one still runs and only the setup that reads no input runs early
    if (ppd::launch_zero_status(dev_status, B, s) != cudaSuccess) return cuda_failed();
    // a bf16 call without a full workspace runs unsplit
    return enqueue_attention_any(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, L, B, H,
                                 T, D, S_max, dt, scale, out, lse, dev_status,
                                 ws_ok ? static_cast<uint8_t *>(workspace) : nullptr, wl, nullptr, s,
                                 true);
}

ppd_status ppd_node_argmax(const float *logits, int B, int T, int V, int32_t *argmax_out,
                           void *workspace, size_t ws_bytes, void *stream)
{
    if (!logits || !argmax_out || B < 1 || T < 1 || V < 1) return PPD_ERR_INVALID_ARG;
    if ((double)B * T * V > 9.0e15 || (double)B * T * 64 > 2147483647.0) return PPD_ERR_INVALID_ARG;
    const WsLayout wl = workspace_layout(1, B, 1, T, 1, V, 0, PPD_BF16);
    if (!workspace || ws_bytes < wl.total || !aligned(workspace, kAlign)) return PPD_ERR_INVALID_ARG;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float *pv = reinterpret_cast<float *>(ws + wl.part_val);
    int32_t *pi = reinterpret_cast<int32_t *>(ws + wl.part_idx);
    const int64_t rows = (int64_t)B * T;
    if (ppd::launch_argmax_partials(logits, rows, V, wl.splits, pv, pi, nullptr, 1.f, nullptr, 0, s) !=
        cudaSuccess)
        return cuda_failed();
    return cuda_status(ppd::launch_argmax_combine(pv, pi, rows, wl.splits, argmax_out, s));
}

ppd_status ppd_accept_path(const int32_t *argmax, const int32_t *cand_tokens,
                           const int32_t *parent, const int32_t *prefix_len,
                           int B, int T, int V, int S_max,
                           int32_t *accept_len, int32_t *path, int32_t *next_token,
                           int32_t *new_prefix_len, int32_t *dev_status, void *stream)
{
    if (!argmax || !cand_tokens || !parent || !prefix_len || !accept_len || !path || !next_token ||
        !new_prefix_len || !dev_status)
        return PPD_ERR_INVALID_ARG;
    if (B < 1 || T < 1 || T > kMaxT || V < 1 || S_max < 0) return PPD_ERR_INVALID_ARG;
    AcceptArgs a{cand_tokens, parent, prefix_len, accept_len, path, next_token, new_prefix_len,
                 dev_status, T, V, S_max};
    return cuda_status(ppd::launch_accept_path(argmax, a, B, static_cast<cudaStream_t>(stream)));
}

ppd_status ppd_kv_compact(void *k_cache, void *v_cache, const void *k_tree, const void *v_tree,
                          const int32_t *path, const int32_t *accept_len,
                          const int32_t *prefix_len, int L, int B, int H, int T, int D,
                          int S_max, ppd_dtype dt, void *stream)
{
    if (!k_cache || !v_cache || !k_tree || !v_tree || !path || !accept_len || !prefix_len)
        return PPD_ERR_INVALID_ARG;
    if (L < 1 || B < 1 || H < 1 || T < 1 || T > kMaxT || D < 1 || S_max < 0) return PPD_ERR_INVALID_ARG;
    if (dt != PPD_BF16 && dt != PPD_F32) return PPD_ERR_INVALID_ARG;
    const int eb = dt == PPD_BF16 ? 2 : 4;
    if ((D * eb) % 16 != 0) return PPD_ERR_UNSUPPORTED;
    if (!aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(k_tree, 16) || !aligned(v_tree, 16))
        return PPD_ERR_INVALID_ARG;
    const size_t lbh = (size_t)L * B * H;
    const size_t nc = lbh * S_max * D * eb, nt = lbh * T * D * eb;
    if (overlaps(k_cache, nc, k_tree, nt) || overlaps(k_cache, nc, v_tree, nt) ||
        overlaps(v_cache, nc, k_tree, nt) || overlaps(v_cache, nc, v_tree, nt) ||
        overlaps(k_cache, nc, v_cache, nc))
        return PPD_ERR_INVALID_ARG;
    return cuda_status(ppd::launch_kv_compact(k_cache, v_cache, k_tree, v_tree, path, accept_len,
                                              prefix_len, L, B, H, T, D, S_max, eb,
                                              static_cast<cudaStream_t>(stream)));
}

ppd_status ppd_verify_step(const void *q, void *k_cache, void *v_cache,
                           const void *k_tree, const void *v_tree,
                           const int32_t *prefix_len, const int32_t *parent,
                           const int32_t *cand_tokens, const float *logits,
                           int L, int B, int H, int T, int D, int V, int S_max, ppd_dtype dt,
                           float scale, float *out, float *lse, int32_t *argmax_out,
                           int32_t *accept_len, int32_t *path, int32_t *next_token,
                           int32_t *new_prefix_len, int32_t *dev_status,
                           void *workspace, size_t ws_bytes, void *stream)
{
    return verify_step_impl(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                            logits, L, B, H, T, D, V, S_max, dt, scale, nullptr, out, lse,
                            argmax_out, accept_len, path, next_token, new_prefix_len, dev_status,
                            workspace, ws_bytes, stream);
}

ppd_status ppd_verify_step_typical(const void *q, void *k_cache, void *v_cache,
                                   const void *k_tree, const void *v_tree,
                                   const int32_t *prefix_len, const int32_t *parent,
                                   const int32_t *cand_tokens, const float *logits,
                                   int L, int B, int H, int T, int D, int V, int S_max,
                                   ppd_dtype dt, float scale, float temperature, float epsilon,
                                   float delta, float *out, float *lse, int32_t *argmax_out,
                                   int32_t *accept_len, int32_t *path, int32_t *next_token,
                                   int32_t *new_prefix_len, int32_t *dev_status,
                                   void *workspace, size_t ws_bytes, void *stream)
{
    if (!typical_params_ok(temperature, epsilon, delta)) return PPD_ERR_INVALID_ARG;
    const TypicalParams typ{temperature, epsilon, delta};
    return verify_step_impl(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                            logits, L, B, H, T, D, V, S_max, dt, scale, &typ, out, lse,
                            argmax_out, accept_len, path, next_token, new_prefix_len, dev_status,
                            workspace, ws_bytes, stream);
}

ppd_status ppd_node_stats(const float *logits, int B, int T, int V, float temperature,
                          int32_t *argmax_out, float *lse_out, float *entropy_out,
                          void *workspace, size_t ws_bytes, void *stream)
{
    if (!logits || !argmax_out || !lse_out || !entropy_out || B < 1 || T < 1 || V < 1)
        return PPD_ERR_INVALID_ARG;
    if (!std::isfinite(temperature) || !(temperature > 0.f) || !std::isfinite(1.f / temperature))
        return PPD_ERR_INVALID_ARG;
    if ((double)B * T * V > 9.0e15 || (double)B * T * 64 > 2147483647.0) return PPD_ERR_INVALID_ARG;
    const WsLayout wl = workspace_layout(1, B, 1, T, 1, V, 0, PPD_BF16);
    if (!workspace || ws_bytes < wl.total || !aligned(workspace, kAlign)) return PPD_ERR_INVALID_ARG;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float *pv = reinterpret_cast<float *>(ws + wl.part_val);
    int32_t *pi = reinterpret_cast<int32_t *>(ws + wl.part_idx);
    float *pst = reinterpret_cast<float *>(ws + wl.part_stats);
    const int64_t rows = (int64_t)B * T;
    if (ppd::launch_argmax_partials(logits, rows, V, wl.splits, pv, pi, pst, temperature, nullptr, 0,
                                    s) != cudaSuccess)
        return cuda_failed();
    return cuda_status(ppd::launch_node_stats_combine(pv, pi, pst, rows, wl.splits, argmax_out,
                                                      lse_out, entropy_out, s));
}

ppd_status ppd_typical_accept(const float *logits, const float *lse, const float *entropy,
                              const int32_t *argmax, const int32_t *cand_tokens,
                              const int32_t *parent, const int32_t *prefix_len, int B, int T,
                              int V, int S_max, float temperature, float epsilon, float delta,
                              int32_t *accept_len, int32_t *path, int32_t *next_token,
                              int32_t *new_prefix_len, int32_t *dev_status, void *stream)
{
    if (!logits || !lse || !entropy || !argmax || !cand_tokens || !parent || !prefix_len ||
        !accept_len || !path || !next_token || !new_prefix_len || !dev_status)
        return PPD_ERR_INVALID_ARG;
    if (B < 1 || T < 1 || T > kMaxT || V < 1 || S_max < 0) return PPD_ERR_INVALID_ARG;
    if (!typical_params_ok(temperature, epsilon, delta)) return PPD_ERR_INVALID_ARG;
    if ((double)B * T * V > 9.0e15) return PPD_ERR_INVALID_ARG;
    AcceptArgs a{cand_tokens, parent, prefix_len, accept_len, path, next_token, new_prefix_len,
                 dev_status, T, V, S_max};
    return cuda_status(ppd::launch_typical_accept(logits, lse, entropy, argmax, a, B, temperature,
                                                  epsilon, delta, static_cast<cudaStream_t>(stream)));
}

// topk [B][n_states][K] int32, kstate [B] int32, then the partial lists
// (values fp32, indices int32) [B][n_states][kNextMaxSplit][K] each, then the
// chain rows' log-sum-exps fp32 [B][n_states][kNextMaxEpt].
static size_t next_part_bytes(int B, int n_states, int K)
{
    return align_up((size_t)B * n_states * ppd::kNextMaxSplit * K * sizeof(int32_t));
}

size_t ppd_next_tree_workspace_bytes(int B, int n_states, int K)
{
    if (B < 1 || n_states < 1 || K < 1) return 0;
    return align_up(align_up((size_t)B * n_states * K * sizeof(int32_t)) + (size_t)B * sizeof(int32_t)) +
           2 * next_part_bytes(B, n_states, K) +
           align_up((size_t)B * n_states * ppd::kNextMaxEpt * sizeof(float));
}

ppd_status ppd_next_tree_ept(const float *logits, const int32_t *parent,
                             const int32_t *cand_tokens, const int32_t *path,
                             const int32_t *accept_len, const int32_t *next_token, int B, int T,
                             int V, int n_states, int T_next, const int32_t *tmpl_parent,
                             const int32_t *tmpl_rank, int K, int n_ept, int ept_mean,
                             int32_t *next_parent, int32_t *next_cand, int32_t *next_state,
                             int32_t *dev_status, void *workspace, size_t ws_bytes, void *stream)
{
    if (!logits || !parent || !cand_tokens || !path || !accept_len || !next_token || !tmpl_parent ||
        !tmpl_rank || !next_parent || !next_cand || !next_state || !dev_status || !workspace)
        return PPD_ERR_INVALID_ARG;
    if (B < 1 || T < 1 || T > kMaxT || V < 1 || n_states < 1 || n_states > 128 || T_next < 1 ||
        T_next > kMaxT || K < 1 || K > V || n_ept < 1 || ept_mean < 0 || ept_mean > 1)
        return PPD_ERR_INVALID_ARG;
    if (K > ppd::kNextMaxK || n_ept > ppd::kNextMaxEpt) return PPD_ERR_UNSUPPORTED;
    if ((double)B * T * V > 9.0e15) return PPD_ERR_INVALID_ARG;
    if (ws_bytes < ppd_next_tree_workspace_bytes(B, n_states, K) || !aligned(workspace, kAlign))
        return PPD_ERR_INVALID_ARG;
    int32_t *topk = static_cast<int32_t *>(workspace);
    int32_t *kstate = reinterpret_cast<int32_t *>(static_cast<char *>(workspace) +
                                                  align_up((size_t)B * n_states * K * sizeof(int32_t)));
    char *parts = static_cast<char *>(workspace) +
                  align_up(align_up((size_t)B * n_states * K * sizeof(int32_t)) + (size_t)B * sizeof(int32_t));
    float *part_val = reinterpret_cast<float *>(parts);
    int32_t *part_idx = reinterpret_cast<int32_t *>(parts + next_part_bytes(B, n_states, K));
    float *lse = reinterpret_cast<float *>(parts + 2 * next_part_bytes(B, n_states, K));
    return cuda_status(ppd::launch_next_tree(
        logits, parent, cand_tokens, path, accept_len, next_token, B, T, V, n_states, T_next,
        tmpl_parent, tmpl_rank, K, n_ept, ept_mean, topk, kstate, part_val, part_idx, lse, num_sms(),
        next_parent, next_cand, next_state, dev_status, static_cast<cudaStream_t>(stream)));
}

ppd_status ppd_next_tree(const float *logits, const int32_t *parent, const int32_t *cand_tokens,
                         const int32_t *path, const int32_t *accept_len, const int32_t *next_token,
                         int B, int T, int V, int n_states, int T_next, const int32_t *tmpl_parent,
                         const int32_t *tmpl_rank, int K, int n_ept, int32_t *next_parent,
                         int32_t *next_cand, int32_t *next_state, int32_t *dev_status,
                         void *workspace, size_t ws_bytes, void *stream)
{
    return ppd_next_tree_ept(logits, parent, cand_tokens, path, accept_len, next_token, B, T, V,
                             n_states, T_next, tmpl_parent, tmpl_rank, K, n_ept, 0, next_parent,
                             next_cand, next_state, dev_status, workspace, ws_bytes, stream);
}

ppd_status ppd_selftest_umma(const void *a, const void *b, float *d, int mode, int N, void *stream)
{
    if (!a || !b || !d || mode < 0 || mode > 3 || N < 16 || N > 256 || N % 16 != 0)
        return PPD_ERR_INVALID_ARG;
    if (mode == 3 && N > 128) return PPD_ERR_INVALID_ARG;
    if (mode != 0 && N % 8 != 0) return PPD_ERR_INVALID_ARG;
    if (!aligned(a, 16) || !aligned(b, 16) || !aligned(d, 4)) return PPD_ERR_INVALID_ARG;
    CUtensorMap ma, mb;
    std::memset(&ma, 0, sizeof ma);
    std::memset(&mb, 0, sizeof mb);
    if (mode == 3) {
        // A is written to TMEM by threads, B to shared memory: no tensor maps
    } else if (mode == 0) {
        if (!encode_2d(&ma, a, 128, 128, 128) || !encode_2d(&mb, b, 128, N, N)) return PPD_ERR_CUDA;
    } else {
        if (!encode_2d(&ma, a, mode == 2 ? 64 : 128, 128, 128)) return PPD_ERR_CUDA;
        mb = ma;
    }
    return cuda_status(ppd::launch_selftest_umma(ma, mb, a, b, d, mode, N, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
