// common.cuh -- device helpers shared by the libsadmm kernels (sm_103a).
//
// Inline PTX wrappers for mbarriers, TMA tensor loads and the 5th-generation
// tensor-core instructions (tcgen05: TMEM allocation, MMA, commit, loads),
// written against the public PTX ISA.  Every spin-wait here is bounded: it
// gives up after kWaitLimitNs of %globaltimer time or when the CTA's abort
// flag is raised, so no kernel can hang the GPU.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "sadmm.h"

#define SADMM_DEV __device__ __forceinline__

namespace sadmm {

// Device-side status codes (written into the library's status word).
constexpr int kDevTimeout = 1;
constexpr int kDevBadIndex = 2;
constexpr int kDevBounds = 3;   // a debug build's index check failed

// A bounded wait gives up after this much wall time.
constexpr unsigned long long kWaitLimitNs = 4000000000ull;  // 4 s

SADMM_DEV uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

SADMM_DEV unsigned long long globaltimer()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// GPU-scope flag operations on global memory (PTX memory model): an acquire
// load, a relaxed store, and an acquire-release fetch-add.
SADMM_DEV int ld_acquire_gpu(const int* p)
{
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

SADMM_DEV void st_relaxed_gpu(int* p, int v)
{
    asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

SADMM_DEV int atom_add_acq_rel_gpu(int* p, int v)
{
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// Programmatic dependent launch (kernels launched with the programmatic stream
// serialization attribute): a kernel may start while the previous kernel of
// its stream is still running; pdl_wait() blocks until that kernel has
// completed and its memory is visible, so it comes before the first read of
// anything an earlier kernel wrote.  pdl_trigger() lets the next kernel of the
// stream be scheduled once every CTA of this one has issued it (or exited).
SADMM_DEV void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
SADMM_DEV void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Host: launch `kern` with programmatic stream serialization (the kernel calls
// pdl_wait() before its first global-memory read).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args... args)
{
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Bits lo .. hi-1 of a word (none when hi <= lo; 0 <= lo and hi <= 31).
SADMM_DEV uint32_t bits_between(int lo, int hi) { return hi > lo ? (1u << hi) - (1u << lo) : 0u; }

// Tap-validity mask of one output pixel whose receptive window starts at
// (it0, ih0, iw0) of a T x H x W input: a bit is set where a tap reads inside
// the input.  One bit per tap t = (kt*KH + kh)*KW + kw when the kernel has at
// most 31 taps (split = 0); otherwise (split = 1) bits 0..15 mark valid rows
// kt*KH + kh and bits 16..30 valid kw.  Bit 31 is never set (the gather
// tables mark padding columns with it).  Each kernel coordinate's valid range
// (0 <= i0 + k < extent) is formed in closed form.
SADMM_DEV uint32_t tap_mask(int it0, int ih0, int iw0, int KT, int KH, int KW, int T, int H, int W, int split)
{
    const int t_lo = max(0, -it0), t_hi = min(KT, T - it0);
    const int h_lo = max(0, -ih0), h_hi = min(KH, H - ih0);
    const int w_lo = max(0, -iw0), w_hi = min(KW, W - iw0);
    const uint32_t cm = bits_between(w_lo, w_hi), hm = bits_between(h_lo, h_hi);
    if (split) {
        uint32_t rm = 0;
        for (int kt = t_lo; kt < t_hi; ++kt) rm |= hm << (kt * KH);
        return rm | (cm << 16);
    }
    uint32_t m = 0;
    for (int kt = t_lo; kt < t_hi; ++kt)
        for (int kh = h_lo; kh < h_hi; ++kh) m |= cm << ((kt * KH + kh) * KW);
    return m;
}

SADMM_DEV void raise_status(int* status, int code)
{
    if (status) atomicCAS(status, 0, code);
}

// Index checks of the debug build (-DSADMM_DEBUG): true when i lies in
// [0, n); otherwise the status word gets kDevBounds and the caller skips the
// access (a load then reads zero).  In the release build every check is the
// constant true and compiles away.
#ifdef SADMM_DEBUG
SADMM_DEV bool dbg_in(long long i, long long n, int* status)
{
    if (i >= 0 && i < n) return true;
    raise_status(status, kDevBounds);
    return false;
}
#else
SADMM_DEV bool dbg_in(long long, long long, int*) { return true; }
#endif

// ---------------------------------------------------------------- mbarrier --

SADMM_DEV void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

SADMM_DEV void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

SADMM_DEV void mbar_arrive(uint64_t* bar)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(smem_u32(bar))
                 : "memory");
}

SADMM_DEV void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(
                     smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

SADMM_DEV bool mbar_try_wait(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// try_wait with a suspend-time hint: a thread whose phase is not complete is
// suspended (it issues nothing) until the phase completes or about `hint_ns`
// pass, instead of spinning on the barrier.
constexpr uint32_t kSuspendHintNs = 1000000;  // 1 ms

SADMM_DEV bool mbar_try_wait_suspend(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(kSuspendHintNs)
        : "memory");
    return ok != 0;
}

// Waits until the phase with the given parity of `bar` has completed.
// Returns false (and raises the abort flag and the status word) when the wait
// runs past `limit_ns`, or false at once when another role aborted.
SADMM_DEV bool mbar_wait_for(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status,
                             unsigned long long limit_ns)
{
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer();
    for (;;) {
        if (mbar_try_wait_suspend(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer() - t0 > limit_ns) {
            *abort_flag = 1;
            raise_status(status, kDevTimeout);
            return false;
        }
    }
}

// mbar_wait_for with the kernels' limit, kWaitLimitNs.
SADMM_DEV bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status)
{
    return mbar_wait_for(bar, parity, abort_flag, status, kWaitLimitNs);
}

// mbar_wait by every lane of a converged warp, with one outcome for all.
SADMM_DEV bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort_flag, int* status)
{
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_flag, status));
}

// --------------------------------------------------------------------- TMA --

// 2-D tiled TMA load of one box into shared memory; completion is signalled
// on `bar` as transaction bytes.  c0 is the innermost (contiguous) coordinate.
SADMM_DEV void tma_load_2d(void* dst, const void* tmap, uint64_t* bar, int c0, int c1)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
        "l"(tmap), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
        : "memory");
}

// 4-D tiled TMA load (coordinates innermost first); completion as for
// tma_load_2d.
SADMM_DEV void tma_load_4d(void* dst, const void* tmap, uint64_t* bar, int c0, int c1, int c2, int c3)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(smem_u32(dst)),
        "l"(tmap), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

SADMM_DEV void tma_prefetch_desc(const void* tmap)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(tmap) : "memory");
}

// Makes this thread's generic-proxy shared-memory writes visible to the async
// proxy (the tensor core reads operands through it).
SADMM_DEV void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ----------------------------------------------------------------- tcgen05 --

// Allocates `ncols` TMEM columns (power of two >= 32); the whole warp calls it.
// The TMEM address is written to shared memory at `dst`.
SADMM_DEV void tmem_alloc(uint32_t* dst, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)),
                 "r"(ncols)
                 : "memory");
}

SADMM_DEV void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

SADMM_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

SADMM_DEV void tc_fence_before()
{
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

SADMM_DEV void tc_fence_after()
{
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulator, one CTA,
// executed by a whole converged warp: the lane elect.sync picks issues (the
// same lane for the same full mask, so its commits track these MMAs).  The
// loop around it then stays warp-uniform: one lane alone forming descriptors
// issued an MMA per 90-130 cycles, against 56 for a 128 x 96 x 16 MMA.
SADMM_DEV void mma_bf16_ss_elect(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p, e;\n\t.reg .b32 l;\n\telect.sync l|e, 0xffffffff;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

// Arrives once on `bar` when every tcgen05 operation the elected lane issued so
// far has completed; executed by a whole converged warp.
SADMM_DEV void mma_commit_elect(uint64_t* bar)
{
    asm volatile(
        "{\n\t.reg .pred e;\n\t.reg .b32 l;\n\telect.sync l|e, 0xffffffff;\n\t"
        "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(smem_u32(bar))
        : "memory");
}

// Each lane of the warp reads 32 consecutive 32-bit TMEM columns of its lane.
SADMM_DEV void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

// 32 lanes x 16 consecutive 32-bit columns: lane i of the warp gets row
// (warp quadrant * 32 + i), columns [col, col + 16).
SADMM_DEV void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15])
        : "r"(taddr));
}

SADMM_DEV void tmem_ld_wait()
{
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major operand stored with the 128-byte
// swizzle: rows of 64 bf16 (128 B), 8-row atoms of 1024 B stacked along M/N
// (stride byte offset 1024).  Tiles start on 1024-byte boundaries; stepping
// along K inside the atom moves the start address by 32 B per 16 elements.
SADMM_DEV uint64_t sdesc_kmajor_sw128(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address, bits [0,14)
    d |= (uint64_t)(16u >> 4) << 16;            // leading byte offset (unused here)
    d |= (uint64_t)(1024u >> 4) << 32;          // stride byte offset, bits [32,46)
    d |= (uint64_t)1 << 46;                     // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;                     // layout: 128-byte swizzle
    return d;
}

// Shared-memory descriptor of a K-major operand without swizzle: core
// matrices of 8 rows x 16 bytes (rows 16 bytes apart), `lbo` bytes between
// core matrices adjacent along K and `sbo` bytes between adjacent groups of 8
// rows.  The start address needs 16-byte alignment only.
SADMM_DEV uint64_t sdesc_kmajor_none(uint32_t saddr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);       // start address, bits [0,14)
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;    // leading byte offset, bits [16,30)
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;    // stride byte offset, bits [32,46)
    d |= (uint64_t)1 << 46;                         // descriptor version for tcgen05
    return d;                                       // layout 0: no swizzle
}

// Instruction descriptor of tcgen05.mma kind::f16: bf16 A and B, both
// K-major, fp32 accumulator, M x N tile.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int m, int n)
{
    return (1u << 4)                        // D format: f32
           | (1u << 7)                      // A format: bf16
           | (1u << 10)                     // B format: bf16
           | ((uint32_t)(n >> 3) << 17)     // N >> 3
           | ((uint32_t)(m >> 4) << 24);    // M >> 4
}

// Byte offset of 16-byte chunk `chunk` (0..7) of row `row` inside a tile
// stored with the 128-byte swizzle (rows of 128 B, tile 1024-byte aligned).
SADMM_DEV uint32_t sw128_offset(uint32_t row, uint32_t chunk)
{
    return row * 128u + ((chunk ^ (row & 7u)) << 4);
}

}  // namespace sadmm
