// ppd_device.cuh -- sm_103a device primitives used by the PPD kernels:
// mbarriers with bounded waits, TMA tensor loads, tcgen05 (TMEM allocation,
// UMMA issue/commit, TMEM loads/stores) and the shared-memory / instruction
// descriptors of the 5th-generation tensor cores, written as inline PTX.
#pragma once

#include "ppd_kernels.h"

#include <cuda.h>
#include <cuda_bf16.h>
#include <cstdint>

#define PPD_DEV __device__ __forceinline__

namespace ppd {

// Internal status codes (mirror ppd_status in include/ppd.h).
enum : int { kOk = 0, kErrInvalidArg = 1, kErrUnsupported = 2, kErrTree = 3,
             kErrCapacity = 4, kErrCuda = 5, kErrTimeout = 6 };


PPD_DEV uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

PPD_DEV uint64_t global_timer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---------------------------------------------------------------- mbarrier

PPD_DEV void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

PPD_DEV void mbar_fence_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

PPD_DEV void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

PPD_DEV void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

PPD_DEV bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

// Wait for the phase with the given parity to complete.  Gives up (and raises
// *abort) after kWaitLimitNs, or as soon as *abort is raised by another thread;
// returns false in both cases.  The caller keeps its control flow unchanged
// either way, so every thread still reaches every named barrier.
PPD_DEV bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort)
{
    const uint32_t a = smem_addr(bar);
    if (mbar_try_wait(a, parity)) return true;
    if (*abort) return false;
    const uint64_t t0 = global_timer();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(a, parity)) return true;
        if ((it & 31u) == 0) {
            if (*abort) return false;
            if (global_timer() - t0 > kWaitLimitNs) {
                *abort = 1;
                return false;
            }
        }
    }
}

// ---------------------------------------------------------------- named barriers

PPD_DEV void named_bar_sync(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Barrier over `nthreads` threads that also returns the OR of `pred`.
PPD_DEV bool named_bar_or(int id, int nthreads, bool pred)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}\n"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
        : "memory");
    return r != 0;
}

// ---------------------------------------------------------------- fences

PPD_DEV void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------- flags between CTAs

PPD_DEV unsigned long long ld_relaxed_gpu(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

PPD_DEV unsigned long long ld_acquire_gpu(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

// A 32-bit load served by L2 (never a stale L1 or texture-cache line).
PPD_DEV int ld_relaxed_gpu_s32(const int *p)
{
    int v;
    asm volatile("ld.relaxed.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

PPD_DEV void st_release_gpu(unsigned long long *p, unsigned long long v)
{
    asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

PPD_DEV void st_relaxed_gpu(unsigned long long *p, unsigned long long v)
{
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

PPD_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
PPD_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32-byte store of eight fp32 values (bit patterns v[0..7]) times `scale` to a
// 32-byte aligned global address: one full sector per thread.
PPD_DEV void st_global_v8(float *dst, const uint32_t *v, float scale)
{
    asm volatile("st.global.v8.f32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(dst),
                 "f"(__uint_as_float(v[0]) * scale), "f"(__uint_as_float(v[1]) * scale),
                 "f"(__uint_as_float(v[2]) * scale), "f"(__uint_as_float(v[3]) * scale),
                 "f"(__uint_as_float(v[4]) * scale), "f"(__uint_as_float(v[5]) * scale),
                 "f"(__uint_as_float(v[6]) * scale), "f"(__uint_as_float(v[7]) * scale)
                 : "memory");
}

// ---------------------------------------------------------------- TMA

PPD_DEV void tma_prefetch_map(const CUtensorMap *map)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}

PPD_DEV uint64_t l2_policy_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

PPD_DEV uint64_t l2_policy_evict_last()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

// 3-D tiled tensor load into shared memory, completion signalled on `bar`
// (complete_tx), with an L2 cache-policy hint.  x must be 16-byte aligned in
// elements*size (every caller passes x in {0, 64} bf16 elements).
PPD_DEV void tma_load_3d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y, int z,
                         uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        ".L2::cache_hint [%0], [%1, {%3, %4, %5}], [%2], %6;" ::"r"(smem_addr(dst)),
        "l"(map), "r"(smem_addr(bar)), "r"(x), "r"(y), "r"(z), "l"(policy)
        : "memory");
}

// Fetch a 3-D tile of a tensor map into L2 only (a hint: no shared memory, no
// completion to wait for).  x must be 16-byte aligned as for tma_load_3d.
PPD_DEV void tma_prefetch_l2_3d(const CUtensorMap *map, int x, int y, int z)
{
    asm volatile("cp.async.bulk.prefetch.tensor.3d.L2.global.tile [%0, {%1, %2, %3}];" ::"l"(map),
                 "r"(x), "r"(y), "r"(z)
                 : "memory");
}

PPD_DEV void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int x, int y)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_addr(dst)),
        "l"(map), "r"(smem_addr(bar)), "r"(x), "r"(y)
        : "memory");
}

// ---------------------------------------------------------------- tcgen05

// Warp-wide: allocate `ncols` TMEM columns (power of two >= 32); the TMEM
// address is written to shared memory at `dst`.
PPD_DEV void tmem_alloc(uint32_t *dst, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(dst)),
                 "r"(ncols)
                 : "memory");
}

PPD_DEV void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

PPD_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr),
                 "r"(ncols)
                 : "memory");
}

// D(tmem) (+)= A(smem) * B(smem), bf16 inputs, fp32 accumulator.
PPD_DEV void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                       uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// D(tmem) (+)= A(tmem) * B(smem), bf16 inputs, fp32 accumulator.  A is M x K
// with row m in TMEM lane m, two consecutive k per 32-bit column (the lower k in
// the low half); a_tmem addresses its first column (lane field 0).
PPD_DEV void umma_bf16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                          uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread is done.
PPD_DEV void umma_commit(uint64_t *bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_addr(bar))
        : "memory");
}

PPD_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
PPD_DEV void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Warp-wide load of 16 consecutive 32-bit TMEM columns; thread i of the warp
// reads lane (32*(warp%4) + i), which must be encoded in taddr's upper half.
PPD_DEV void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

PPD_DEV void tmem_st16(uint32_t taddr, const uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),
        "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]),
        "r"(r[14]), "r"(r[15])
        : "memory");
}

// ---------------------------------------------------------------- descriptors

// Shared-memory matrix descriptor for tcgen05.mma with the 128-byte swizzle.
// Operand tiles are built from 1024-byte atoms: 8 rows of 128 bytes, the
// 16-byte chunks of row r XOR-permuted by (r mod 8) -- exactly what TMA writes
// with CU_TENSOR_MAP_SWIZZLE_128B into a 1024-byte aligned buffer.
//   K-major operand (K contiguous): lbo unused, sbo = byte stride between
//     consecutive 8-row groups along M/N; advancing K by 16 elements moves the
//     start address by 32 bytes inside the atom.
//   M/N-major operand (M or N contiguous): lbo = byte stride between
//     consecutive 64-element groups along M/N, sbo = byte stride between
//     consecutive 8-row groups along K.
PPD_DEV uint64_t make_smem_desc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;  // swizzle mode: 128-byte
    return d;
}

// The descriptor of the same operand `bytes` further on (bytes a multiple of 16):
// only the 14-bit start-address field (16-byte units) changes, and shared
// memory addresses stay below 256 KB, so the field never carries.
PPD_DEV uint64_t desc_advance(uint64_t desc, uint32_t bytes)
{
    return desc + (uint64_t)(bytes >> 4);
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 A and B, fp32 D,
// shape M x N, operand majorness (0 = K-major, 1 = M/N-major).
__host__ __device__ constexpr uint32_t make_idesc_bf16(int M, int N, int a_mn_major,
                                                       int b_mn_major)
{
    return (1u << 4)                                 // D format: f32
           | (1u << 7)                               // A format: bf16
           | (1u << 10)                              // B format: bf16
           | ((uint32_t)a_mn_major << 15)            // A major
           | ((uint32_t)b_mn_major << 16)            // B major
           | ((uint32_t)(N >> 3) << 17)              // N / 8
           | ((uint32_t)(M >> 4) << 24);             // M / 16
}

// Byte offset of element (row, col) of a bf16 tile stored in 128-byte-swizzled
// atoms whose 64-column groups are `group_stride` bytes apart (row < 8*k).
PPD_DEV uint32_t sw128_offset(int row, int col, uint32_t group_stride)
{
    const int group = col >> 6;
    const int chunk = (col & 63) >> 3;
    return (uint32_t)group * group_stride + (uint32_t)(row >> 3) * 1024u +
           (uint32_t)(row & 7) * 128u + (uint32_t)((chunk ^ (row & 7)) << 4) +
           (uint32_t)((col & 7) * 2);
}

// ---------------------------------------------------------------- math

PPD_DEV float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

PPD_DEV float lg2(float x)
{
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

PPD_DEV float rcp(float x)
{
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Maximum of v over the 32 lanes of a warp (every lane gets it).
PPD_DEV float warp_max(float v)
{
    float r;
    asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
    return r;
}

// Reduce 16 per-lane columns over the 32 lanes of a warp.  On return lane L
// holds the reduction of column (L >> 1) over all lanes (lanes 2c and 2c+1
// agree).  16 shuffles for 16 columns.
template <class Op>
PPD_DEV float warp_transpose_reduce16(float (&v)[16], int lane, Op op)
{
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const bool up = lane & 16;
        const float send = up ? v[i] : v[i + 8];
        const float keep = up ? v[i + 8] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 16));
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const bool up = lane & 8;
        const float send = up ? v[i] : v[i + 4];
        const float keep = up ? v[i + 4] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 8));
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const bool up = lane & 4;
        const float send = up ? v[i] : v[i + 2];
        const float keep = up ? v[i + 2] : v[i];
        v[i] = op(keep, __shfl_xor_sync(0xffffffffu, send, 4));
    }
    {
        const bool up = lane & 2;
        const float send = up ? v[0] : v[1];
        const float keep = up ? v[1] : v[0];
        v[0] = op(keep, __shfl_xor_sync(0xffffffffu, send, 2));
    }
    v[0] = op(v[0], __shfl_xor_sync(0xffffffffu, v[0], 1));
    return v[0];
}

struct OpMax {
    PPD_DEV float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct OpAdd {
    PPD_DEV float operator()(float a, float b) const { return a + b; }
};

}  // namespace ppd
