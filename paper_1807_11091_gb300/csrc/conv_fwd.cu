// conv_fwd.cu -- pruned CONV forward as an implicit GEMM on the sm_103a tensor
// cores (Sec. 3: after filter-wise (row) and channel-/shape-wise (column)
// pruning the layer is a smaller full GEMM).
//
//   D[m, i] = sum_{j < K'} A[m, j] * Wp[i, j]
//   A[m, j] = x[n, g*Cg + c_j, ot*st-pt+kt_j, oh*sh-ph+kh_j, ow*sw-pw+kw_j]
//
// m runs over output pixels (N*OT*OH*OW), i over the kept filters of conv group
// g, j over the kept (channel, tap) columns.  Pixels are the MMA M side (128 per
// tile, one TMEM lane each), kept filters the N side (bn <= 256 per tile), so a
// gathered pixel tile is reused by every kept filter of the tile.
//
// One persistent CTA per SM, warp-specialised (896 threads):
//   warp 0      TMA producer: 64-column x bn-row boxes of Wp (128-byte swizzle)
//   warp 1      TMEM allocator and MMA issuer (tcgen05.mma kind::f16, bf16 in,
//               fp32 accumulate, 128 x n x 16 per instruction)
//   warps 4-11  epilogue (two warps per TMEM lane quadrant): tcgen05.ld of the accumulator (lane = pixel), bias,
//               ReLU, coalesced stores to the NCHW output (consecutive lanes
//               write consecutive pixels of one filter plane), and zero-fill of
//               the pruned filters' planes for the tile's pixels
//   warps 12-27 gather: four threads per pixel of the tile, each building two
//               16-byte K-major chunks of A through the gather table, with zero
//               fill outside the input, into the 128-byte-swizzled stage buffer
// Shared-memory stages are guarded by mbarriers; the accumulator is double
// buffered in TMEM so the epilogue of one tile overlaps the MMAs of the next.
#include <cuda.h>
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kBM = 128;           // pixels per tile
constexpr int kBK = 64;            // GEMM columns per stage
constexpr int kGatherWarps = 16;
constexpr int kEpiWarps = 8;
constexpr int kThreads = (4 + kEpiWarps + kGatherWarps) * 32;
constexpr int kGatherThreads = kGatherWarps * 32;
constexpr int kGatherGroups = kGatherThreads / kBM;     // threads per pixel
constexpr int kChunksPerThread = 8 / kGatherGroups;     // 16-byte chunks of a stage row per thread
static_assert(kGatherThreads % kBM == 0 && 8 % kGatherGroups == 0, "gather threads must split a 64-column row evenly");
constexpr int kATileBytes = kBM * kBK * 2;  // 16 KB
constexpr int kMaxStages = 4;
constexpr int kMaxGroups = 64;
constexpr int kTouchAhead = 2;  // stages ahead whose input lines the gather touches
constexpr int kSmemTail = 10240;  // barriers, TMEM address, counts, epilogue tables

struct ConvArgs {
    const __nv_bfloat16* x;
    void* y;
    const float* bias;
    const uint2* gather;  // [k_pad] {channel/tap offset in x, tap bits}
    const int2* stage_chan;  // [k_pad/64] first and last channel of each stage
    const int* rowmap;
    const int* zeromap;
    const int* counts;
    int* status;
    long long M;      // N * plane
    long long x_chw;  // elements per input image
    long long thw;    // elements per input channel
    long long units;  // m_tiles * groups * upairs
    int hw, W, H, T;
    int F, groups, Cg, Fg;
    int OW, OHW, plane;
    int st, sh, sw, pt, ph, pw;
    int KT, KH, KW;
    int nks;  // k_pad / 64
    int bn, n_tiles, n_pad;
    int nacc;      // filter tiles per unit (TMEM accumulators sharing one A tile)
    int upairs;    // units per (pixel tile, group): ceil(n_tiles / nacc)
    int acc_bufs;  // accumulator sets in TMEM (2: the epilogue overlaps the next unit's MMAs)
    int stages;
    int k_pad;
    int n_cols;          // K' (columns past it are padding)
    int split_mask;      // tap-mask encoding: 0 one bit per tap, 1 row bits + kw bits
    uint32_t full_mask;  // the mask of a pixel whose every tap is inside the input
    int tmem_stride;
    int tmem_cols;
    int relu;
};

// Unit u covers filter tiles p*nacc .. p*nacc+nacc-1 of conv group g for pixel
// tile mt.
SADMM_DEV void decode_unit(const ConvArgs& a, long long u, int& p, int& g, long long& mt)
{
    p = (int)(u % a.upairs);
    const long long t = u / a.upairs;
    g = (int)(t % a.groups);
    mt = t / a.groups;
}

// Tap-validity mask of one output pixel: a bit is set where a tap reads inside
// the input.  One bit per tap t = (kt*KH + kh)*KW + kw when the kernel has at
// most 31 taps; otherwise bits 0..15 mark valid rows kt*KH + kh and bits
// 16..30 valid kw.  Bit 31 is never set (it marks padding columns).
SADMM_DEV uint32_t pixel_mask(const ConvArgs& a, int it0, int ih0, int iw0)
{
    uint32_t rm = 0, cm = 0;
    for (int kt = 0; kt < a.KT; ++kt) {
        const bool vt = (unsigned)(it0 + kt) < (unsigned)a.T;
        for (int kh = 0; kh < a.KH; ++kh)
            if (vt && (unsigned)(ih0 + kh) < (unsigned)a.H) rm |= 1u << (kt * a.KH + kh);
    }
    for (int kw = 0; kw < a.KW; ++kw)
        if ((unsigned)(iw0 + kw) < (unsigned)a.W) cm |= 1u << kw;
    if (a.split_mask) return rm | (cm << 16);
    uint32_t m = 0;
    for (int r = 0; r < a.KT * a.KH; ++r)
        if (rm & (1u << r)) m |= cm << (r * a.KW);
    return m;
}

// Gather entry e = {offset in x, tap bits}: the column reads inside the input
// for a pixel of mask M when every tap bit of the entry is set in M.
SADMM_DEV bool tap_ok(uint32_t bits, uint32_t M) { return (M & bits) == bits; }

// Input lines one tile reads, for touching them ahead of the gather: image n,
// depth slices [t0, t0+nt), rows [r0, r0+nr) (clamped), and this thread's
// share: line `li` of (channel, slice) pair `pr` of a stage.
struct TouchPlan {
    const char* base;  // x[n, g*Cg, 0, 0, 0] plus this thread's (slice, first row, line) offset
    int pc;            // channel offset of this thread's pair from the stage's first channel
    int end_off;       // bytes from the plane's range start to its end (exclusive)
    int line_off;      // this thread's line within the range (0 = the range start)
};

SADMM_DEV TouchPlan touch_plan(const ConvArgs& a, long long u, int t)
{
    TouchPlan tp{nullptr, 0, 0, 0};
    int nt_, g;
    long long mt;
    decode_unit(a, u, nt_, g, mt);
    const long long m0 = mt * kBM;
    if (m0 >= a.M) return tp;
    const long long n = m0 / a.plane;
    long long m1 = min(m0 + kBM - 1, a.M - 1);
    m1 = min(m1, (n + 1) * (long long)a.plane - 1);
    const int p0 = (int)(m0 - n * a.plane), p1 = (int)(m1 - n * a.plane);
    const int ot0 = p0 / a.OHW, ot1 = p1 / a.OHW;
    int oh0 = 0, oh1 = a.OHW / a.OW - 1;
    if (ot0 == ot1) {
        oh0 = (p0 - ot0 * a.OHW) / a.OW;
        oh1 = (p1 - ot1 * a.OHW) / a.OW;
    }
    const int r0 = max(0, oh0 * a.sh - a.ph), r1 = min(a.H - 1, oh1 * a.sh - a.ph + a.KH - 1);
    const int t0 = max(0, ot0 * a.st - a.pt), t1 = min(a.T - 1, ot1 * a.st - a.pt + a.KT - 1);
    if (r1 < r0 || t1 < t0) return tp;
    // this thread's share: line li of (channel, slice) pair pr of a stage
    const int nt2 = t1 - t0 + 1, nr = r1 - r0 + 1;
    const int per = (2 * nr * a.W + 127) / 128 + 1;  // lines a (channel, slice) range can touch
    const int pr = t / per, li = t - pr * per;
    tp.pc = pr / nt2;
    const int it = t0 + pr % nt2;
    tp.base = reinterpret_cast<const char*>(a.x) +
              2 * (n * a.x_chw + (long long)g * a.Cg * a.thw + (long long)it * a.hw + (long long)r0 * a.W);
    tp.end_off = 2 * nr * a.W;
    tp.line_off = li;
    return tp;
}

SADMM_DEV void touch_stage(const ConvArgs& a, const TouchPlan& tp, int ks)
{
    if (!tp.base || ks >= a.nks) return;
    const int2 cr = __ldg(a.stage_chan + ks);
    if (cr.x + tp.pc > cr.y) return;
    const char* start = tp.base + 2 * (long long)(cr.x + tp.pc) * a.thw;
    const char* addr = reinterpret_cast<const char*>(((reinterpret_cast<uintptr_t>(start) >> 7) + tp.line_off) << 7);
    if (addr >= start + tp.end_off) return;
    if (addr < start) addr = start;
    asm volatile("{\n\t.reg .b16 t;\n\tld.global.nc.b16 t, [%0];\n\t}" ::"l"(addr));
}

// Branch-free conditional gather: the 16-bit element at p when every tap bit
// of `bits` is set in the pixel mask M, else 0 (a predicated load).
SADMM_DEV uint32_t ldg_u16_if(const unsigned short* p, uint32_t bits, uint32_t M)
{
    uint32_t v;
    asm("{\n\t.reg .pred q;\n\t.reg .b32 t;\n\t"
        "and.b32 t, %2, %3;\n\t"
        "setp.eq.b32 q, t, %3;\n\t"
        "mov.b32 %0, 0;\n\t"
        "@q ld.global.nc.u16 %0, [%1];\n\t}"
        : "=r"(v)
        : "l"(p), "r"(M), "r"(bits));
    return v;
}

template <bool OUT_BF16>
__global__ void __launch_bounds__(kThreads, 1)
    k_conv_fwd(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ ConvArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = a.stages;
    const uint32_t b_bytes = (uint32_t)a.bn * 128u;      // one Wp box (bn rows x 64 columns)
    const uint32_t bstage = b_bytes * (uint32_t)a.nacc;  // a B stage holds nacc boxes
    uint8_t* sA = smem;
    uint8_t* sB = smem + (size_t)S * kATileBytes;
    uint2* s_table = reinterpret_cast<uint2*>(sB + (size_t)S * bstage);
    uint64_t* bars = reinterpret_cast<uint64_t*>(s_table + a.k_pad);
    uint64_t* full_a = bars;
    uint64_t* full_b = bars + S;
    uint64_t* empty = bars + 2 * S;
    uint64_t* acc_full = bars + 3 * S;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* drain = acc_empty + 2;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
    int* s_counts = reinterpret_cast<int*>(tmem_holder + 2);
    int* s_eoff = s_counts + 2 * kMaxGroups;                   // [2][512] output-plane offsets
    float* s_ebias = reinterpret_cast<float*>(s_eoff + 1024);  // [2][512] biases

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full_a[s], kGatherThreads);
            mbar_init(&full_b[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < a.acc_bufs; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], kEpiWarps * 32);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    for (int i = threadIdx.x; i < 2 * a.groups; i += blockDim.x) s_counts[i] = a.counts[i];
    {
        // the gather table is the same for every tile: keep it in shared memory
        const uint4* src = reinterpret_cast<const uint4*>(a.gather);
        uint4* dst = reinterpret_cast<uint4*>(s_table);
        for (int i = threadIdx.x; i < a.k_pad / 2; i += blockDim.x) dst[i] = __ldg(src + i);
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tmap);
    if (warp == 1) {
        tmem_alloc(tmem_holder, (uint32_t)a.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer (Wp)
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            uint32_t issued_parity[kMaxStages];
            uint32_t issued_mask = 0;
            bool ok = true;
            for (long long u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
                int p, g;
                long long mt;
                decode_unit(a, u, p, g, mt);
                const int nt0 = p * a.nacc;
                if (s_counts[2 * g] <= nt0 * a.bn) continue;
                int nbox = 0;  // filter tiles of this unit with kept rows
                for (int i = 0; i < a.nacc; ++i)
                    if (nt0 + i < a.n_tiles && s_counts[2 * g] > (nt0 + i) * a.bn) nbox = i + 1;
                const int row0 = g * a.n_pad + nt0 * a.bn;
                for (int ks = 0; ks < a.nks; ++ks) {
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) { ok = false; break; }
                    mbar_arrive_expect_tx(&full_b[s], b_bytes * (uint32_t)nbox);
                    for (int i = 0; i < nbox; ++i)
                        tma_load_2d(sB + (size_t)s * bstage + (size_t)i * b_bytes, &tmap, &full_b[s], ks * kBK,
                                    row0 + i * a.bn);
                    issued_parity[s] = ph;
                    issued_mask |= 1u << s;
                    if (++s == S) { s = 0; ph ^= 1u; }
                }
            }
            // Every box this thread issued has landed before the CTA retires
            // (normally already true: the MMA consumed them).
            for (int q = 0; q < S; ++q) {
                if (!(issued_mask & (1u << q))) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full_b[q], issued_parity[q]) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            int ab = 0;
            uint32_t acc_ph = 0;
            bool ok = true;
            for (long long u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
                int p, g;
                long long mt;
                decode_unit(a, u, p, g, mt);
                const int cnt = s_counts[2 * g] - p * a.nacc * a.bn;  // kept rows from the unit's first tile
                if (cnt <= 0) continue;
                // one accumulator per filter tile with kept rows, N rounded up to 16
                const int rows1 = (a.nacc == 2 && p * 2 + 1 < a.n_tiles) ? min(a.bn, cnt - a.bn) : 0;
                const uint32_t idesc0 = idesc_bf16_f32(kBM, min(a.bn, (cnt + 15) & ~15));
                const uint32_t idesc1 = idesc_bf16_f32(kBM, min(a.bn, (max(rows1, 16) + 15) & ~15));
                const bool two = rows1 > 0;
                if (!mbar_wait(&acc_empty[ab], acc_ph ^ 1u, abort_flag, a.status)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(ab * a.nacc * a.tmem_stride);
                for (int ks = 0; ks < a.nks; ++ks) {
                    if (!mbar_wait(&full_a[s], ph, abort_flag, a.status) ||
                        !mbar_wait(&full_b[s], ph, abort_flag, a.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + (size_t)s * kATileBytes);
                    const uint32_t b0 = smem_u32(sB + (size_t)s * bstage);
                    // The issuing thread is on the critical path: straight-line
                    // code, descriptors in registers.
                    if (!two) {
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk)
                            mma_bf16_ss(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32),
                                        idesc0, (ks | kk) != 0 ? 1u : 0u);
                    } else {
                        const uint32_t d1 = d_tmem + (uint32_t)a.tmem_stride;
                        const uint32_t b1 = b0 + b_bytes;
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk) {
                            const uint64_t adesc = sdesc_kmajor_sw128(a0 + kk * 32);
                            const uint32_t acc = (ks | kk) != 0 ? 1u : 0u;
                            mma_bf16_ss(d_tmem, adesc, sdesc_kmajor_sw128(b0 + kk * 32), idesc0, acc);
                            mma_bf16_ss(d1, adesc, sdesc_kmajor_sw128(b1 + kk * 32), idesc1, acc);
                        }
                    }
                    mma_commit(&empty[s]);
                    if (++s == S) { s = 0; ph ^= 1u; }
                }
                if (!ok) break;
                mma_commit(&acc_full[ab]);
                if (++ab == a.acc_bufs) { ab = 0; acc_ph ^= 1u; }
            }
            // Every MMA this thread issued has completed before TMEM is freed.
            mma_commit(drain);
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
        }
        __syncwarp();
    } else if (warp >= 4 && warp < 4 + kEpiWarps) {
        // --------------------------------------------------------- epilogue
        // kEpiWarps / 4 warps share each TMEM lane quadrant and split its
        // 32-column chunks.  Per unit, the output-plane offset and bias of every
        // packed row go to shared memory before the accumulator wait, so the
        // store loop reads them with broadcast loads.
        constexpr int kHalves = kEpiWarps / 4;
        const int q = warp & 3;  // TMEM lane quadrant this warp may access
        const int h = (warp - 4) >> 2;
        const int et = threadIdx.x - 4 * 32;  // 0 .. kEpiWarps*32-1
        const int row = q * 32 + lane;
        int ab = 0;
        uint32_t acc_ph = 0;
        int ub = 0;  // double-buffered per-unit tables
        for (long long u = blockIdx.x; u < a.units; u += gridDim.x) {
            int p, g;
            long long mt;
            decode_unit(a, u, p, g, mt);
            const int nt0 = p * a.nacc;
            const int cnt = s_counts[2 * g] - nt0 * a.bn;  // kept rows from the unit's first tile
            const long long m = mt * kBM + row;
            const bool valid = m < a.M;
            const long long n_img = valid ? m / a.plane : 0;
            const long long pix = valid ? m - n_img * a.plane : 0;
            float* yf = reinterpret_cast<float*>(a.y) + (n_img * (long long)a.F * a.plane + pix);
            __nv_bfloat16* yh = reinterpret_cast<__nv_bfloat16*>(a.y) + (n_img * (long long)a.F * a.plane + pix);
            int* u_off = s_eoff + ub * 512;
            float* u_bias = s_ebias + ub * 512;
            if (cnt > 0) {
                // column i of the unit = row i % bn of filter tile nt0 + i / bn
                const int* rmap = a.rowmap + (long long)g * a.n_pad + (long long)nt0 * a.bn;
                const int ncol = min(a.nacc, a.n_tiles - nt0) * a.bn;
                for (int i = et; i < ncol; i += kEpiWarps * 32) {
                    const int f = __ldg(rmap + i);
                    u_off[i] = f >= 0 ? f * a.plane : 0;
                    u_bias[i] = (f >= 0 && a.bias) ? __ldg(a.bias + f) : 0.0f;
                }
            }
            asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
            if (cnt > 0) {
                // warp-uniform outcome: the TMEM loads below are .sync.aligned
                if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[ab], acc_ph, abort_flag, a.status))) break;
                tc_fence_after();
                for (int ti = 0; ti < a.nacc && nt0 + ti < a.n_tiles; ++ti) {
                    const int nrows = min(a.bn, cnt - ti * a.bn);
                    if (nrows <= 0) break;
                    const uint32_t taddr = tmem_base + (uint32_t)((ab * a.nacc + ti) * a.tmem_stride) +
                                           ((uint32_t)(q * 32) << 16);
                    const int* t_off = u_off + ti * a.bn;
                    const float* t_bias = u_bias + ti * a.bn;
                    for (int c0 = 32 * h; c0 < nrows; c0 += 32 * kHalves) {
                        uint32_t r[32];
                        tmem_ld_32x32b_x32(taddr + (uint32_t)c0, r);
                        tmem_ld_wait();
                        if (valid) {
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                if (c0 + j < nrows) {
                                    float v = __uint_as_float(r[j]) + t_bias[c0 + j];
                                    if (a.relu) v = fmaxf(v, 0.0f);
                                    if (OUT_BF16)
                                        yh[t_off[c0 + j]] = __float2bfloat16_rn(v);
                                    else
                                        __stcs(yf + t_off[c0 + j], v);
                                }
                            }
                        }
                    }
                }
                tc_fence_before();
                mbar_arrive(&acc_empty[ab]);
                if (++ab == a.acc_bufs) { ab = 0; acc_ph ^= 1u; }
            }
            if (p == 0) {
                // pruned filters of this conv group: their planes are zero
                const int zc = s_counts[2 * g + 1];
                const int* zmap = a.zeromap + (long long)g * a.Fg;
                for (int z0 = 32 * h; z0 < zc; z0 += 32 * kHalves) {
                    const int zo = (z0 + lane < zc) ? __ldg(zmap + z0 + lane) * a.plane : 0;
                    const int zn = min(32, zc - z0);
                    for (int j = 0; j < zn; ++j) {
                        const int off = __shfl_sync(0xffffffffu, zo, j);
                        if (valid) {
                            if (OUT_BF16)
                                yh[off] = __float2bfloat16_rn(0.0f);
                            else
                                __stcs(yf + off, 0.0f);
                        }
                    }
                }
            }
            ub ^= 1;
        }
    } else if (warp >= 4 + kEpiWarps) {
        // ----------------------------------------------------------- gather
        const int gt = threadIdx.x - (4 + kEpiWarps) * 32;
        const int prow = gt & (kBM - 1);
        const int chunk0 = gt >> 7;  // this thread builds chunks chunk0 + kGatherGroups * i
        const unsigned short* xs = reinterpret_cast<const unsigned short*>(a.x);
        int s = 0;
        uint32_t ph = 0;
        bool ok = true;
        int touched = 0;  // leading stages of the current unit already touched
        for (long long u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
            int p, g;
            long long mt;
            decode_unit(a, u, p, g, mt);
            if (s_counts[2 * g] <= p * a.nacc * a.bn) {
                touched = 0;
                continue;
            }
            const TouchPlan tp_cur = touch_plan(a, u, gt);
            const TouchPlan tp_next = touch_plan(a, u + gridDim.x, gt);
            for (int q = touched; q < kTouchAhead; ++q) touch_stage(a, tp_cur, q);
            const long long m = mt * kBM + prow;
            uint32_t M = 0;
            const unsigned short* xb = xs;
            if (m < a.M) {
                const long long n_img = m / a.plane;
                const int p = (int)(m - n_img * a.plane);
                const int ot = p / a.OHW;
                const int r2 = p - ot * a.OHW;
                const int oh = r2 / a.OW;
                const int ow = r2 - oh * a.OW;
                const int it0 = ot * a.st - a.pt, ih0 = oh * a.sh - a.ph, iw0 = ow * a.sw - a.pw;
                M = pixel_mask(a, it0, ih0, iw0);
                xb = xs + (n_img * a.x_chw + (long long)g * a.Cg * a.thw + (long long)it0 * a.hw +
                           (long long)ih0 * a.W + iw0);
            }
            // Every lane's pixel sees every tap: no bounds test is needed.
            const bool interior = __all_sync(0xffffffffu, M == a.full_mask);
            for (int ks = 0; ks < a.nks; ++ks) {
                // Land the input lines of the stage kTouchAhead ahead (of the
                // next tile near the end of this one) in L1.
                if (ks + kTouchAhead < a.nks)
                    touch_stage(a, tp_cur, ks + kTouchAhead);
                else
                    touch_stage(a, tp_next, ks + kTouchAhead - a.nks);
                // Issue every load of this thread's columns first (they read
                // only x), then wait for the stage buffer and store.
                const uint2* te = s_table + (size_t)ks * kBK;
                uint32_t v[8 * kChunksPerThread];
                // two table entries per 16-byte shared-memory load
                const uint4* te4 = reinterpret_cast<const uint4*>(te);
                if (interior && (ks + 1) * kBK <= a.n_cols) {
#pragma unroll
                    for (int ci = 0; ci < kChunksPerThread; ++ci) {
                        const int c = chunk0 + kGatherGroups * ci;
#pragma unroll
                        for (int e = 0; e < 8; e += 2) {
                            const uint4 t = te4[(c * 8 + e) >> 1];
                            v[ci * 8 + e] = __ldg(xb + (int)t.x);
                            v[ci * 8 + e + 1] = __ldg(xb + (int)t.z);
                        }
                    }
                } else {
#pragma unroll
                    for (int ci = 0; ci < kChunksPerThread; ++ci) {
                        const int c = chunk0 + kGatherGroups * ci;
#pragma unroll
                        for (int e = 0; e < 8; e += 2) {
                            const uint4 t = te4[(c * 8 + e) >> 1];
                            v[ci * 8 + e] = ldg_u16_if(xb + (int)t.x, t.y, M);
                            v[ci * 8 + e + 1] = ldg_u16_if(xb + (int)t.z, t.w, M);
                        }
                    }
                }
                if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) { ok = false; break; }
                uint8_t* tile = sA + (size_t)s * kATileBytes;
#pragma unroll
                for (int ci = 0; ci < kChunksPerThread; ++ci) {
                    const int c = chunk0 + kGatherGroups * ci;
                    const uint32_t* q = v + ci * 8;
                    *reinterpret_cast<uint4*>(tile + sw128_offset((uint32_t)prow, (uint32_t)c)) =
                        make_uint4(__byte_perm(q[0], q[1], 0x5410), __byte_perm(q[2], q[3], 0x5410),
                                   __byte_perm(q[4], q[5], 0x5410), __byte_perm(q[6], q[7], 0x5410));
                }
                fence_proxy_async_smem();
                mbar_arrive(&full_a[s]);
                if (++s == S) { s = 0; ph ^= 1u; }
            }
            touched = min(kTouchAhead, a.nks);
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, (uint32_t)a.tmem_cols);
    }
}

template <bool OUT_BF16>
cudaError_t launch(const CUtensorMap& map, const ConvArgs& a, int grid, size_t smem, cudaStream_t s)
{
    auto kern = k_conv_fwd<OUT_BF16>;
    static int configured_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_dev != dev) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
        if (e != cudaSuccess) return e;
        configured_dev = dev;
    }
    kern<<<grid, kThreads, smem, s>>>(map, a);
    return cudaGetLastError();
}

}  // namespace

sadmm_status launch_conv_fwd(const sadmm_plan* plan, const Geometry& g, const void* x, const float* bias,
                             int relu, void* y, int ydt, cudaStream_t s)
{
    if (g.groups > kMaxGroups) return SADMM_EUNSUPPORTED;
    const char* base = static_cast<const char*>(plan->dev);
    ConvArgs a;
    memset(&a, 0, sizeof(a));
    a.x = static_cast<const __nv_bfloat16*>(x);
    a.y = y;
    a.bias = bias;
    a.gather = reinterpret_cast<const uint2*>(base + plan->off_gather);
    a.stage_chan = reinterpret_cast<const int2*>(a.gather + plan->k_pad);
    a.rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    a.zeromap = reinterpret_cast<const int*>(base + plan->off_zeromap);
    a.counts = reinterpret_cast<const int*>(base + plan->off_counts);
    a.status = device_status_ptr();
    a.M = g.m;
    a.x_chw = g.c * g.t * g.h * g.w;
    a.thw = g.t * g.h * g.w;
    a.hw = (int)(g.h * g.w);
    a.W = (int)g.w;
    a.H = (int)g.h;
    a.T = (int)g.t;
    a.F = (int)g.f;
    a.groups = (int)g.groups;
    a.Cg = (int)g.cg;
    a.Fg = (int)g.fg;
    a.OW = (int)g.ow;
    a.OHW = (int)(g.oh * g.ow);
    a.plane = (int)g.plane;
    a.st = (int)g.st;
    a.sh = (int)g.sh;
    a.sw = (int)g.sw;
    a.pt = (int)g.pt;
    a.ph = (int)g.ph;
    a.pw = (int)g.pw;
    a.KT = (int)g.kt;
    a.KH = (int)g.kh;
    a.KW = (int)g.kw;
    a.nks = plan->k_pad / kBK;
    a.bn = plan->bn;
    a.n_tiles = plan->n_tiles;
    a.nacc = plan->n_tiles >= 2 ? 2 : 1;
    a.upairs = (plan->n_tiles + a.nacc - 1) / a.nacc;
    a.n_pad = plan->n_pad;
    a.relu = relu ? 1 : 0;
    const long long m_tiles = (g.m + kBM - 1) / kBM;
    a.units = m_tiles * g.groups * a.upairs;

    a.k_pad = plan->k_pad;
    a.n_cols = plan->n_cols;
    a.split_mask = tap_mask_mode(g);
    if (a.split_mask)
        a.full_mask = ((1u << (g.kt * g.kh)) - 1u) | (((1u << g.kw) - 1u) << 16);
    else
        a.full_mask = (uint32_t)((1ull << g.taps) - 1ull);
    const int stage_bytes = kATileBytes + a.nacc * plan->bn * 128;
    const int table_bytes = plan->k_pad * 8;
    const int budget = 232448 - 1024 - kSmemTail - table_bytes;
    // At most kMaxStages: what shared memory leaves over serves as L1 for x.
    a.stages = budget / stage_bytes;
    if (a.stages > kMaxStages) a.stages = kMaxStages;
    if (a.stages < 2) return SADMM_EUNSUPPORTED;
    a.tmem_stride = (plan->bn + 31) & ~31;
    a.acc_bufs = (2 * a.nacc * a.tmem_stride <= 512) ? 2 : 1;
    int cols = 32;
    while (cols < a.acc_bufs * a.nacc * a.tmem_stride) cols <<= 1;
    a.tmem_cols = cols;
    const size_t smem = 1024 + (size_t)a.stages * stage_bytes + table_bytes + kSmemTail;

    long long grid = device_sm_count();
    if (grid > a.units) grid = a.units;
    if (grid < 1) grid = 1;

    CUtensorMap map;
    memcpy(&map, plan->tmap, sizeof(map));
    const cudaError_t e = (ydt == SADMM_BF16) ? launch<true>(map, a, (int)grid, smem, s)
                                              : launch<false>(map, a, (int)grid, smem, s);
    return e == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
