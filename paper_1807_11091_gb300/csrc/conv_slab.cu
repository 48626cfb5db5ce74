// conv_slab.cu -- the input-slab forward of a pruned CONV layer whose kept
// channels keep every column (Sec. 3: the pruned layer is a smaller full GEMM;
// here the layers with no column pruning, or whole channels pruned, and few
// input channels -- a network's first layer, which the paper keeps whole).
//
// k_slab_input rewrites x as a space-to-depth copy xs[n][chunk][pixel][8]:
// block pixel (hb, wb) of image n holds, for kept channel ci and phase
// (a, b) < (sh, sw), slab channel cc = (ci*sh + a)*sw + b (8 per chunk) =
// x[n][chan[ci]][hb*sh + a - ph][wb*sw + b - pw], zero outside.  Output pixel
// (oh, ow) and kernel tap (kh, kw) = (r*sh + a, q*sw + b) read block pixel
// (oh + r, ow + q), phase (a, b): the layer becomes a stride-1 R x Q conv over
// cs slab channels (R = ceil(KH/sh), Q = ceil(KW/sw)).  k_slab_input_rows
// writes the same copy when sw divides 8 (each input row's offset and
// validity formed once per row, not per element).
//
// k_conv_slab: GEMM row i of tile t of image n is block pixel p = 128t + i of
// that image's output grid laid out in rows of Wb = OW + Q - 1 block pixels
// (row oh = p / Wb, column ow = p % Wb; columns past OW and rows past OH are
// computed and dropped).  Block tap (r, q) of row i reads block pixel
// p + r*Wb + q, so a tile needs the sp = 128 + (R-1)*Wb + Q-1 consecutive
// block pixels from 128t on -- its slab, one TMA box of every chunk,
// [chunk][pixel][8 channels] in shared memory.  The A operand of tap (r, q)
// is that slab shifted by r*Wb + q pixels: K-major core matrices of 8 pixels
// x 8 channels (16-byte rows), no swizzle, so any pixel offset is a valid
// start.  B (the kept filters' weights in slab column order, tap-major) stays
// resident in shared memory, 128-byte swizzled.
//   warp 0      TMA: the weights once, then one slab per tile
//   warp 1      TMEM allocator and MMA issuer (R*Q*cs/16 MMAs of
//               128 x bn x 16 per tile, fp32 accumulator in TMEM, two sets)
//   warps 2-9   epilogue: tcgen05.ld (lane = GEMM row), bias, ReLU, stores
//               to the NCHW output, zero planes of the pruned filters
#include <cuda.h>
#include <string.h>

#include "common.cuh"
#include "conv_common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kSlabWarps = 10;
constexpr int kSlabThreads = kSlabWarps * 32;
constexpr int kSlabEpiWarps = 8;        // warps 2..9: two per TMEM lane quadrant (warp % 4)
constexpr int kMaxSlabStages = 4;
constexpr int kSlabTables = 2 * 256 * 4;  // plane offset and bias of each kept row
constexpr int kSlabZcap = 1024;           // pruned filters whose plane offsets sit in shared memory
constexpr int kSlabBars = 256;            // barriers, TMEM address, abort flag
constexpr int kSlabSmemLimit = 232448;
constexpr int kSlabMaxSteps = 128;  // MMAs per tile whose descriptor offsets travel in the parameters

struct SlabArgs {
    void* y;
    const float* bias;
    const int* rowmap;   // packed row -> filter (-1: padding)
    const int* zeromap;  // pruned filters, ascending
    const int* counts;   // [kept, pruned]
    int* status;
    long long y_total;  // elements of y (the debug build's store checks)
    int F, OH, OW, plane;
    int Wb, MT, units;     // block-pixel row width, tiles per image, tiles in all
    FastDiv mt_div, wb_div;
    int sp, R, Q, ksteps;  // slab pixels, block taps, MMAs of 16 columns per tap
    int bn, nbox;          // MMA N, 64-column weight boxes
    int stages, stage_bytes, stage_stride;
    int tmem_stride, tmem_cols;
    int relu;
    int nsteps;                     // MMAs per tile (R * Q * ksteps)
    uint2 steps[kSlabMaxSteps];     // per MMA: A start (16-byte units from the slab), B start (from the weights)
};

struct XsArgs {
    int C, H, W, sh, sw, ph, pw;
    int nck, cs, Hb, Wb, pimg;
    long long x_total, xs_total;  // elements of x and of the copy (the debug build's index checks)
    int* status;
};

// Thread (tx, ty) of block (bw, bh, n) writes every chunk's 16-byte vector
// (8 slab channels) of block pixel (hb, wb) = (4*bh + ty, 64*bw + tx) of image
// n; the loads of two chunks (16) are in flight together.  The channel and
// phase of each slab channel come from a table decoded once per block in
// shared memory.
constexpr int kXsPix = 64;   // block pixels of a block row per block (threadIdx.x)
constexpr int kXsRows = 4;   // block rows per block (threadIdx.y)
__global__ void __launch_bounds__(kXsPix * kXsRows) k_slab_input(const __nv_bfloat16* __restrict__ x,
                                                                 const int* __restrict__ chan, const XsArgs b,
                                                                 __nv_bfloat16* __restrict__ xs)
{
    __shared__ int4 s_dec[64];  // per slab channel: {channel plane offset (-1: zero), a - ph, b - pw, 0}
    pdl_wait();  // after the kernel before it in the stream
    const int n = blockIdx.z;
    const int tid = threadIdx.y * kXsPix + threadIdx.x;
    if (tid < b.cs) {
        const int cc = tid;
        const int ci = cc / (b.sh * b.sw);
        const int ch = ci < b.nck ? (chan ? __ldg(chan + ci) : ci) : -1;
        s_dec[cc] = make_int4(ch >= 0 ? ch * b.H * b.W : -1, (cc / b.sw) % b.sh - b.ph, cc % b.sw - b.pw, 0);
    }
    __syncthreads();
    const int chunks = b.cs / 8;
    if (blockIdx.x == 0 && blockIdx.y == 0) {
        // the pixels past Hb*Wb up to pimg (fewer than 8 per chunk row) are zero:
        // they are read by the GEMM rows past the output, and the weight gradient
        // multiplies them by those rows' zero dZ
        const int pad = b.pimg - b.Hb * b.Wb;
        for (int v = tid; v < chunks * pad; v += kXsPix * kXsRows) {
            const int k = v / pad, j = v - k * pad;
            const long long o = (((long long)n * chunks + k) * b.pimg + (long long)b.Hb * b.Wb + j) * 8;
            if (dbg_in(o + 7, b.xs_total, b.status)) *reinterpret_cast<uint4*>(xs + o) = make_uint4(0u, 0u, 0u, 0u);
        }
    }
    const int wb = blockIdx.x * kXsPix + threadIdx.x;
    const int hb = blockIdx.y * kXsRows + threadIdx.y;
    if (wb >= b.Wb || hb >= b.Hb) return;
    const unsigned short* xi = reinterpret_cast<const unsigned short*>(x) + (long long)n * b.C * b.H * b.W;
    const int ih0 = hb * b.sh, iw0 = wb * b.sw;
    __nv_bfloat16* dst0 = xs + ((long long)n * chunks * b.pimg + (long long)hb * b.Wb + wb) * 8;
#pragma unroll 2
    for (int k = 0; k < chunks; ++k) {
        uint32_t h[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int4 d = s_dec[8 * k + e];
            const int ih = ih0 + d.y, iw = iw0 + d.z;
            h[e] = (d.x >= 0 && (unsigned)ih < (unsigned)b.H && (unsigned)iw < (unsigned)b.W &&
                    dbg_in(xi - reinterpret_cast<const unsigned short*>(x) + d.x + ih * b.W + iw, b.x_total, b.status))
                       ? (uint32_t)__ldg(xi + d.x + ih * b.W + iw)
                       : 0u;
        }
        if (dbg_in(dst0 - xs + (long long)k * b.pimg * 8 + 7, b.xs_total, b.status))
            *reinterpret_cast<uint4*>(dst0 + (long long)k * b.pimg * 8) =
                make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16), h[6] | (h[7] << 16));
    }
}

// The same copy when the column stride SW divides 8: a chunk's 8 slab
// channels cc = (ci*sh + a)*SW + b are then 8/SW input rows rho = ci*sh + a
// (channel chan[ci], row hb*sh + a - ph) of SW consecutive columns
// wb*SW + b - pw each.  A thread forms each row's offset and validity once
// and each column's validity once, so an element costs a predicated load at
// a constant offset from its row (the generic kernel decodes every element).
// Thread t of block (bx, n) writes block pixel p = 256*bx + t of image n
// (hb = p / Wb, wb = p % Wb): no lanes idle at the end of a block row.
constexpr int kXsFlat = 256;  // block pixels per block
template <int SW>
__global__ void __launch_bounds__(kXsFlat) k_slab_input_rows(const __nv_bfloat16* __restrict__ x,
                                                            const int* __restrict__ chan, const XsArgs b,
                                                            const FastDiv wb_div, __nv_bfloat16* __restrict__ xs)
{
    constexpr int kRows = 8 / SW;  // input rows per chunk
    __shared__ int2 s_row[64];     // per row rho < cs/SW: {channel plane offset (-1: zero), a - ph}
    pdl_wait();  // after the kernel before it in the stream
    const int n = blockIdx.y;
    const int tid = threadIdx.x;
    if (tid < b.cs / SW) {
        const int ci = tid / b.sh;
        const int ch = ci < b.nck ? (chan ? __ldg(chan + ci) : ci) : -1;
        s_row[tid] = make_int2(ch >= 0 ? ch * b.H * b.W : -1, tid - ci * b.sh - b.ph);
    }
    __syncthreads();
    const int chunks = b.cs / 8;
    const int npix = b.Hb * b.Wb;
    if (blockIdx.x == 0) {
        // the pixels past Hb*Wb up to pimg (fewer than 8 per chunk row) are zero:
        // they are read by the GEMM rows past the output, and the weight gradient
        // multiplies them by those rows' zero dZ
        const int pad = b.pimg - npix;
        for (int v = tid; v < chunks * pad; v += kXsFlat) {
            const int k = v / pad, j = v - k * pad;
            const long long o = (((long long)n * chunks + k) * b.pimg + npix + j) * 8;
            if (dbg_in(o + 7, b.xs_total, b.status)) *reinterpret_cast<uint4*>(xs + o) = make_uint4(0u, 0u, 0u, 0u);
        }
    }
    const int p = blockIdx.x * kXsFlat + tid;
    if (p >= npix) return;
    const int hb = (int)fdiv((uint32_t)p, wb_div);
    const int wb = p - hb * b.Wb;
    const int ih0 = hb * b.sh, iw0 = wb * SW - b.pw;
    bool col_ok[SW];
#pragma unroll
    for (int c = 0; c < SW; ++c) col_ok[c] = (unsigned)(iw0 + c) < (unsigned)b.W;
    const long long img = (long long)n * b.C * b.H * b.W;
    const unsigned short* xi = reinterpret_cast<const unsigned short*>(x);
    __nv_bfloat16* dst0 = xs + ((long long)n * chunks * b.pimg + p) * 8;
#pragma unroll 2
    for (int k = 0; k < chunks; ++k) {
        uint32_t h[8];
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            const int2 s = s_row[k * kRows + r];
            const int ih = ih0 + s.y;
            const bool row_ok = s.x >= 0 && (unsigned)ih < (unsigned)b.H;
            // element offset of column 0 of this row (only read where the row and column are inside x)
            const long long e0 = img + s.x + (long long)ih * b.W + iw0;
#pragma unroll
            for (int c = 0; c < SW; ++c)
                h[r * SW + c] = (row_ok && col_ok[c] && dbg_in(e0 + c, b.x_total, b.status))
                                    ? (uint32_t)__ldg(xi + e0 + c)
                                    : 0u;
        }
        if (dbg_in(dst0 - xs + (long long)k * b.pimg * 8 + 7, b.xs_total, b.status))
            *reinterpret_cast<uint4*>(dst0 + (long long)k * b.pimg * 8) =
                make_uint4(h[0] | (h[1] << 16), h[2] | (h[3] << 16), h[4] | (h[5] << 16), h[6] | (h[7] << 16));
    }
}

template <bool OUT_BF16>
__global__ void __launch_bounds__(kSlabThreads, 1)
    k_conv_slab(const __grid_constant__ CUtensorMap tw, const __grid_constant__ CUtensorMap tx,
                const __grid_constant__ SlabArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t bbox = (uint32_t)a.bn * 128u;  // one 64-column box of the weights
    uint8_t* sB = smem;
    uint8_t* sA = sB + (size_t)a.nbox * bbox;  // 1024-aligned: bbox is a multiple of 2048
    int* t_off = reinterpret_cast<int*>(sA + (size_t)a.stages * a.stage_stride);
    float* t_bias = reinterpret_cast<float*>(t_off + 256);
    int* z_off = reinterpret_cast<int*>(t_bias + 256);  // [kSlabZcap] plane offsets of pruned filters
    uint64_t* bars = reinterpret_cast<uint64_t*>(z_off + kSlabZcap);
    uint64_t* full = bars;
    uint64_t* empty = bars + kMaxSlabStages;
    uint64_t* acc_full = bars + 2 * kMaxSlabStages;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* b_full = acc_empty + 2;
    uint64_t* drain = b_full + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kMaxSlabStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], kSlabEpiWarps);
        }
        mbar_init(b_full, 1);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, (uint32_t)a.tmem_cols);
        tmem_relinquish();
    }
    // Nothing above reads global memory: it overlaps the previous kernel's tail.
    pdl_wait();
    pdl_trigger();
    for (int i = threadIdx.x; i < a.bn; i += blockDim.x) {
        const int f = __ldg(a.rowmap + i);
        t_off[i] = f >= 0 ? f * a.plane : 0;
        t_bias[i] = (f >= 0 && a.bias) ? __ldg(a.bias + f) : 0.0f;
    }
    const int zc = min(__ldg(a.counts + 1), kSlabZcap);
    for (int z = threadIdx.x; z < zc; z += blockDim.x) z_off[z] = __ldg(a.zeromap + z) * a.plane;
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tw);
        tma_prefetch_desc(&tx);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            mbar_arrive_expect_tx(b_full, bbox * (uint32_t)a.nbox);
            for (int i = 0; i < a.nbox; ++i) tma_load_2d(sB + (size_t)i * bbox, &tw, b_full, i * 64, 0);
            int s = 0;
            uint32_t ph = 0;
            uint32_t issued_parity[kMaxSlabStages];
            uint32_t issued_mask = 0;
            for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
                const int n = (int)fdiv((uint32_t)u, a.mt_div);
                const int t = u - n * a.MT;
                if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) break;
                mbar_arrive_expect_tx(&full[s], (uint32_t)a.stage_bytes);
                // the tile's slab: block pixels 128t .. 128t+sp-1 (octets 16t ..), every chunk
                tma_load_4d(sA + (size_t)s * a.stage_stride, &tx, &full[s], 0, t * 16, 0, n);
                issued_parity[s] = ph;
                issued_mask |= 1u << s;
                if (++s == a.stages) { s = 0; ph ^= 1u; }
            }
            // every copy this thread issued has landed before the CTA retires
            for (int q = 0; q < a.stages; ++q) {
                if (!(issued_mask & (1u << q))) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full[q], issued_parity[q]) && globaltimer() - t0 < kWaitLimitNs) {}
            }
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(b_full, 0) && globaltimer() - t0 < kWaitLimitNs) {}
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        // The whole warp runs the loop, so the descriptors stay warp-uniform;
        // one elected lane issues the MMAs and the commits that track them.
        bool ok = mbar_wait_warp(b_full, 0, abort_flag, a.status);
        const uint32_t idesc = idesc_bf16_f32(128, a.bn);
        const uint64_t ad0 = sdesc_kmajor_none(smem_u32(sA), (uint32_t)a.sp * 16u, 128u);
        const uint64_t bd0 = sdesc_kmajor_sw128(smem_u32(sB));
        const uint32_t ahi = (uint32_t)(ad0 >> 32), bhi = (uint32_t)(bd0 >> 32), blo = (uint32_t)bd0;
        int s = 0, ab = 0;
        uint32_t ph = 0, acc_ph = 0;
        for (int u = blockIdx.x; ok && u < a.units; u += gridDim.x) {
            if (!mbar_wait_warp(&acc_empty[ab], acc_ph ^ 1u, abort_flag, a.status)) break;
            tc_fence_after();
            if (!mbar_wait_warp(&full[s], ph, abort_flag, a.status)) break;
            tc_fence_after();
            const uint32_t d = tmem_base + (uint32_t)(ab * a.tmem_stride);
            // The low descriptor word starts with the start-address field (the
            // shared address / 16, below 2^14), so offsets in 16-byte units add to it.
            const uint32_t alo = (uint32_t)ad0 + ((uint32_t)(s * a.stage_stride) >> 4);
#pragma unroll 4
            for (int st = 0; st < a.nsteps; ++st) {
                const uint2 e = a.steps[st];
                mma_bf16_ss_elect(d, ((uint64_t)ahi << 32) | (alo + e.x), ((uint64_t)bhi << 32) | (blo + e.y), idesc,
                                  st > 0 ? 1u : 0u);
            }
            mma_commit_elect(&empty[s]);
            mma_commit_elect(&acc_full[ab]);
            if (++s == a.stages) { s = 0; ph ^= 1u; }
            if (++ab == 2) { ab = 0; acc_ph ^= 1u; }
        }
        // Every MMA the elected lane issued has completed before TMEM is freed.
        mma_commit_elect(drain);
        if (lane == 0) {
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------- epilogue
        const int q = warp & 3;          // TMEM lane quadrant this warp may access
        const int h = (warp - 2) >> 2;   // which of the quadrant's two warps
        const int row = q * 32 + lane;
        const int kept = __ldg(a.counts), pruned = __ldg(a.counts + 1);
        const int nch = (kept + kEpiCols - 1) / kEpiCols;
        int ab = 0;
        uint32_t acc_ph = 0;
        bool alive = true;
        for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
            const int n = (int)fdiv((uint32_t)u, a.mt_div);
            const int t = u - n * a.MT;
            const int p = t * 128 + row;
            const int oh = (int)fdiv((uint32_t)p, a.wb_div);
            const int ow = p - oh * a.Wb;
            const bool valid = oh < a.OH && ow < a.OW;
            const long long pix = (long long)n * a.F * a.plane + (long long)oh * a.OW + ow;
            float* yf = reinterpret_cast<float*>(a.y) + pix;
            __nv_bfloat16* yh = reinterpret_cast<__nv_bfloat16*>(a.y) + pix;
            const YCheck yc{pix, a.y_total, a.status};
            // pruned filters' planes: zero, while the tile's MMAs run
            if (alive && valid) {
                for (int z = h; z < pruned; z += 2) {
                    const long long off = z < kSlabZcap ? z_off[z] : (long long)__ldg(a.zeromap + z) * a.plane;
                    if (!y_ok(yc, off)) continue;
                    if (OUT_BF16)
                        yh[off] = __float2bfloat16_rn(0.0f);
                    else
                        __stcs(yf + off, 0.0f);
                }
            }
            // warp-uniform outcome: the TMEM loads below are .sync.aligned
            if (alive && !__all_sync(0xffffffffu, mbar_wait(&acc_full[ab], acc_ph, abort_flag, a.status)))
                alive = false;
            if (alive) {
                tc_fence_after();
                const uint32_t taddr = tmem_base + (uint32_t)(ab * a.tmem_stride) + ((uint32_t)(q * 32) << 16);
                for (int k = h; k < nch; k += 2) {
                    const int c0 = k * kEpiCols;
                    uint32_t r[kEpiCols];
                    tmem_ld_32x32b_x16(taddr + (uint32_t)c0, r);
                    tmem_ld_wait();
                    float v[kEpiCols];
#pragma unroll
                    for (int j = 0; j < kEpiCols; ++j) v[j] = __uint_as_float(r[j]);
                    if (valid) store_cols<OUT_BF16>(v, c0, kept, t_off, t_bias, a.relu, yf, yh, yc);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_empty[ab]);
            }
            if (++ab == 2) { ab = 0; acc_ph ^= 1u; }
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, (uint32_t)a.tmem_cols);
    }
}

int slab_fixed_bytes(int bn, int kpad_s)
{
    return 1024 + (kpad_s / 64) * bn * 128 + kSlabTables + kSlabZcap * 4 + kSlabBars;
}
int slab_stage_stride(int cs, int sp) { return (int)round_up((long long)cs * sp * 2, 1024); }

template <bool OUT_BF16>
cudaError_t launch_slab(const CUtensorMap& tw, const CUtensorMap& tx, const SlabArgs& a, int grid, size_t smem,
                        cudaStream_t s)
{
    auto kern = k_conv_slab<OUT_BF16>;
    static int configured_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_dev != dev) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSlabSmemLimit);
        if (e != cudaSuccess) return e;
        configured_dev = dev;
    }
    return launch_pdl(kern, dim3((unsigned)grid), dim3(kSlabThreads), smem, s, tw, tx, a);
}

}  // namespace

int slab_stages(int bn, int kpad_s, int cs, int sp)
{
    if (bn < 16 || bn > 256 || bn % 16 || kpad_s % 64 || cs % 16 || sp % 8 || kpad_s / 16 > kSlabMaxSteps) return 0;
    const long long room = (long long)kSlabSmemLimit - slab_fixed_bytes(bn, kpad_s);
    if (room <= 0) return 0;
    const long long st = room / slab_stage_stride(cs, sp);
    return (int)(st > kMaxSlabStages ? kMaxSlabStages : st);
}

sadmm_status launch_conv_slab(const sadmm_plan* plan, const Geometry& g, const void* x, const float* bias, int relu,
                              void* y, int ydt, int phase, cudaStream_t s)
{
    const int stages = slab_stages(plan->bn, plan->xs_kpad, plan->xs_cs, plan->xs_sp);
    if (stages < 2 || plan->n_tiles != 1 || g.groups != 1 || plan->xs_cs > 64 || plan->xs_cs % 16 ||
        (long long)(plan->colkind == SADMM_COL_CHANNEL ? plan->n_colgroups : g.c) * g.sh * g.sw > plan->xs_cs)
        return SADMM_EINVAL;  // not a slab plan
    const char* base = static_cast<const char*>(plan->dev);
    const long long mt = ((long long)g.oh * plan->xs_wb + 127) / 128;
    const long long units = g.n * mt;
    if (units >= (1ll << 31) - (1ll << 20) || (long long)plan->xs_hb * plan->xs_wb >= (1ll << 31) - 256)
        return SADMM_EUNSUPPORTED;
    XsArgs b;
    b.C = (int)g.c;
    b.H = (int)g.h;
    b.W = (int)g.w;
    b.sh = (int)g.sh;
    b.sw = (int)g.sw;
    b.ph = (int)g.ph;
    b.pw = (int)g.pw;
    b.nck = plan->colkind == SADMM_COL_CHANNEL ? plan->n_colgroups : (int)g.c;
    b.cs = plan->xs_cs;
    b.Hb = plan->xs_hb;
    b.Wb = plan->xs_wb;
    b.pimg = plan->xs_pimg;
    b.x_total = g.n * g.c * g.h * g.w;
    b.xs_total = g.n * (long long)(plan->xs_cs / 8) * plan->xs_pimg * 8;
    b.status = device_status_ptr();
    // without channel pruning the kept channels are 0 .. C-1: the pass then
    // reads nothing sadmm_pack writes (it may overlap the layer's pack)
    const int* chan = plan->colkind == SADMM_COL_CHANNEL
                          ? reinterpret_cast<const int*>(base + plan->off_scol) + plan->xs_kpad
                          : nullptr;
    __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(const_cast<char*>(base) + plan->off_xs);
    if (phase != SADMM_FWD_REST) {
        const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
        const dim3 flat((unsigned)((plan->xs_hb * plan->xs_wb + kXsFlat - 1) / kXsFlat), (unsigned)g.n);
        const FastDiv wdiv = make_fastdiv((uint32_t)plan->xs_wb);
        cudaError_t e;
        switch (g.sw) {
        case 1: e = launch_pdl(k_slab_input_rows<1>, flat, dim3(kXsFlat), 0, s, xb, chan, b, wdiv, xs); break;
        case 2: e = launch_pdl(k_slab_input_rows<2>, flat, dim3(kXsFlat), 0, s, xb, chan, b, wdiv, xs); break;
        case 4: e = launch_pdl(k_slab_input_rows<4>, flat, dim3(kXsFlat), 0, s, xb, chan, b, wdiv, xs); break;
        case 8: e = launch_pdl(k_slab_input_rows<8>, flat, dim3(kXsFlat), 0, s, xb, chan, b, wdiv, xs); break;
        default:
            e = launch_pdl(k_slab_input,
                           dim3((unsigned)((plan->xs_wb + kXsPix - 1) / kXsPix),
                                (unsigned)((plan->xs_hb + kXsRows - 1) / kXsRows), (unsigned)g.n),
                           dim3(kXsPix, kXsRows), 0, s, xb, chan, b, xs);
        }
        if (e != cudaSuccess) return SADMM_ECUDA;
    }

    if (phase == SADMM_FWD_INPUT) return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
    SlabArgs a;
    memset(&a, 0, sizeof(a));
    a.y = y;
    a.bias = bias;
    a.rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    a.zeromap = reinterpret_cast<const int*>(base + plan->off_zeromap);
    a.counts = reinterpret_cast<const int*>(base + plan->off_counts);
    a.status = device_status_ptr();
    a.y_total = g.n * g.f * g.plane;
    a.F = (int)g.f;
    a.OH = (int)g.oh;
    a.OW = (int)g.ow;
    a.plane = (int)g.plane;
    a.Wb = plan->xs_wb;
    a.MT = (int)mt;
    a.units = (int)units;
    a.mt_div = make_fastdiv((uint32_t)mt);
    a.wb_div = make_fastdiv((uint32_t)plan->xs_wb);
    a.sp = plan->xs_sp;
    a.R = plan->xs_r;
    a.Q = plan->xs_q;
    a.ksteps = plan->xs_cs / 16;
    a.bn = plan->bn;
    a.nbox = plan->xs_kpad / 64;
    a.stages = stages;
    a.stage_bytes = plan->xs_cs * plan->xs_sp * 2;
    a.stage_stride = slab_stage_stride(plan->xs_cs, plan->xs_sp);
    a.tmem_stride = (int)round_up(plan->bn, 32);
    int cols = 32;
    while (cols < 2 * a.tmem_stride) cols <<= 1;
    a.tmem_cols = cols;
    a.relu = relu ? 1 : 0;
    a.nsteps = a.R * a.Q * a.ksteps;
    {
        int st = 0;
        for (int r = 0; r < a.R; ++r)
            for (int q = 0; q < a.Q; ++q)
                for (int j = 0; j < a.ksteps; ++j, ++st)
                    a.steps[st] = make_uint2((uint32_t)(r * a.Wb + q) + (uint32_t)j * (uint32_t)a.sp * 2u,
                                             (uint32_t)(st >> 2) * (uint32_t)a.bn * 8u + (uint32_t)(st & 3) * 2u);
    }
    const size_t smem = (size_t)slab_fixed_bytes(a.bn, plan->xs_kpad) + (size_t)stages * a.stage_stride;
    long long grid = plan->ctas > 0 ? plan->ctas : device_sm_count();
    if (grid > units) grid = units;
    if (grid < 1) grid = 1;
    CUtensorMap tw, tx;
    memcpy(&tw, plan->tmap_ws, sizeof(tw));
    memcpy(&tx, plan->tmap_xs, sizeof(tx));
    const cudaError_t e = (ydt == SADMM_BF16) ? launch_slab<true>(tw, tx, a, (int)grid, smem, s)
                                              : launch_slab<false>(tw, tx, a, (int)grid, smem, s);
    return e == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
