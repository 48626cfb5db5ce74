// bwd_slab.cu -- weight gradient of an input-slab plan (the first layer of a
// network, kept whole: masked retraining, Sec. 4) without an im2col copy.
//
// With dZ = dY * [y > 0] and the forward's space-to-depth input xs (slab
// channel cc of block pixel q; see conv_slab.cu), slab column j = (tap, cc),
// tap = (r, q):
//   dWs[i][j] = sum over images and output pixels p of dZ[i][p] * xs[cc][p + r*Wb + q]
// where p runs over the block-pixel grid of the output (rows of Wb = OW+Q-1;
// dZ is zero on the columns past OW and the rows past OH).  This is a GEMM
// with the kept filters on the MMA's M side, the slab channels of one tap on
// its N side and pixels on K: the A operand is a tile of dZ (128 filter rows x
// 128 grid pixels, K-major, 128-byte swizzle, by TMA from a grid-layout copy
// of dZ), the B operand the tile's slab shifted by r*Wb + q pixels, read
// MN-major (core matrices of 8 channels x 8 pixels, 16-byte rows: the slab
// layout itself).  Each CTA accumulates all of its tiles in TMEM (R*Q*cs
// columns, at most 512), writes one fp32 slice [bn][R*Q*cs], and a second
// kernel adds the slices in CTA order into dW through the slab column map.
//   warp 0      TMA: per tile the slab (every chunk) and two 64-pixel boxes of dZ
//   warp 1      TMEM allocator and MMA issuer (R*Q*(128/16) MMAs per tile)
//   warps 2-9   at the end: tcgen05.ld of the accumulator, stores to the slice
#include <cuda.h>
#include <cudaTypedefs.h>
#include <string.h>

#include <algorithm>

#include "common.cuh"
#include "conv_common.cuh"
#include "internal.h"

namespace sadmm {

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn();  // pack.cu

namespace {

constexpr int kWgWarps = 10;
constexpr int kWgThreads = kWgWarps * 32;
constexpr int kWgMaxStages = 4;
constexpr int kWgDzBox = 128 * 128;      // one 64-pixel box of 128 dZ rows (bf16)
constexpr int kWgSmemLimit = 232448;
constexpr long long kWgMaxCtas = 160;    // slices the workspace holds (grid <= this)

struct WgArgs {
    int units, MT;          // tiles in all, tiles per image
    FastDiv mt_div;
    int sp, R, Q, Wb;       // slab pixels, block taps, block-pixel row width
    int cs, nchunks;        // slab channels (MMA N per tap), 8-channel chunks
    int bn, cols;           // dZ rows per image, slab columns R*Q*cs
    int stages, stage_stride, slab_bytes;
    float* slices;          // [grid][bn][cols]
    int* status;
};

// dZ in the output's block-pixel grid: dzt[n][i][p], p < MT*128, for the
// plan's packed rows i < bn (zero past the kept ones and off the output).
__global__ void __launch_bounds__(256) k_slab_dzt(const __nv_bfloat16* __restrict__ dy, const void* y, int ydt,
                                                  int relu, const int* __restrict__ rowmap, int kept, int bn, int F,
                                                  int OH, int OW, int Wb, int pg, __nv_bfloat16* __restrict__ dzt)
{
    pdl_wait();  // after the kernel before it in the stream
    const int p = blockIdx.x * blockDim.x + threadIdx.x;
    const int i = blockIdx.y, n = blockIdx.z;
    if (p >= pg) return;
    const int oh = p / Wb, ow = p - oh * Wb;
    float v = 0.0f;
    if (i < kept && oh < OH && ow < OW) {
        const int f = __ldg(rowmap + i);
        if (f >= 0) {
            const size_t off = (((size_t)n * F + f) * OH + oh) * OW + ow;
            v = __bfloat162float(dy[off]);
            if (relu) {
                const float yv = ydt == SADMM_BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(y)[off])
                                                   : static_cast<const float*>(y)[off];
                if (!(yv > 0.0f)) v = 0.0f;
            }
        }
    }
    dzt[((size_t)n * bn + i) * pg + p] = __float2bfloat16_rn(v);
}

// Instruction descriptor: bf16 A (K-major) and B (MN-major), fp32 D, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32_bmn(int m, int n)
{
    return idesc_bf16_f32(m, n) | (1u << 16);  // B transposed: MN-major
}

__global__ void __launch_bounds__(kWgThreads, 1)
    k_wgrad_slab(const __grid_constant__ CUtensorMap tx, const __grid_constant__ CUtensorMap td,
                 const __grid_constant__ WgArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + (size_t)a.stages * a.stage_stride);
    uint64_t* full = bars;
    uint64_t* empty = bars + kWgMaxStages;
    uint64_t* acc_full = bars + 2 * kWgMaxStages;
    uint64_t* drain = acc_full + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kWgMaxStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, 512u);
        tmem_relinquish();
    }
    pdl_wait();
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tx);
        tma_prefetch_desc(&td);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            uint32_t issued_parity[kWgMaxStages];
            uint32_t issued_mask = 0;
            for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
                const int n = (int)fdiv((uint32_t)u, a.mt_div);
                const int t = u - n * a.MT;
                if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) break;
                uint8_t* st = smem + (size_t)s * a.stage_stride;
                mbar_arrive_expect_tx(&full[s], (uint32_t)a.slab_bytes + 2u * kWgDzBox);
                // the slab: block pixels 128t .. 128t+sp-1 (octets 16t ..), every chunk
                tma_load_4d(st, &tx, &full[s], 0, t * 16, 0, n);
                // dZ rows n*bn .. +127, grid pixels 128t .. +63 and +64 .. +127
                uint8_t* dz = st + (size_t)a.stage_stride - 2 * kWgDzBox;
                tma_load_2d(dz, &td, &full[s], t * 128, n * a.bn);
                tma_load_2d(dz + kWgDzBox, &td, &full[s], t * 128 + 64, n * a.bn);
                issued_parity[s] = ph;
                issued_mask |= 1u << s;
                if (++s == a.stages) { s = 0; ph ^= 1u; }
            }
            for (int q = 0; q < a.stages; ++q) {
                if (!(issued_mask & (1u << q))) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full[q], issued_parity[q]) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        // The whole warp runs the loop (warp-uniform descriptors); one elected
        // lane issues the MMAs and the commits that track them.
        {
            const uint32_t idesc = idesc_bf16_f32_bmn(128, a.cs);
            const uint32_t sbo = (uint32_t)a.sp * 16u;  // next 8-channel chunk (along N)
            int s = 0;
            uint32_t ph = 0;
            bool first = true, ok = true;
            for (int u = blockIdx.x; u < a.units; u += gridDim.x) {
                if (!mbar_wait_warp(&full[s], ph, abort_flag, a.status)) { ok = false; break; }
                tc_fence_after();
                const uint32_t x0 = smem_u32(smem + (size_t)s * a.stage_stride);
                const uint32_t d0 = x0 + (uint32_t)a.stage_stride - 2u * kWgDzBox;
                for (int r = 0; r < a.R; ++r) {
                    for (int q = 0; q < a.Q; ++q) {
                        const uint32_t xt = x0 + (uint32_t)(r * a.Wb + q) * 16u;
                        const uint32_t d = tmem_base + (uint32_t)((r * a.Q + q) * a.cs);
#pragma unroll
                        for (int kk = 0; kk < 8; ++kk) {
                            // 16 grid pixels: dZ K-major (swizzled box kk / 4), slab rows MN-major
                            const uint64_t adesc =
                                sdesc_kmajor_sw128(d0 + (uint32_t)(kk >> 2) * kWgDzBox + (uint32_t)(kk & 3) * 32u);
                            const uint64_t bdesc = sdesc_kmajor_none(xt + (uint32_t)kk * 256u, 128u, sbo);
                            mma_bf16_ss_elect(d, adesc, bdesc, idesc, (first && kk == 0) ? 0u : 1u);
                        }
                    }
                }
                first = false;
                mma_commit_elect(&empty[s]);
                if (++s == a.stages) { s = 0; ph ^= 1u; }
            }
            if (ok) mma_commit_elect(acc_full);
            mma_commit_elect(drain);
            if (lane == 0) {
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------- epilogue (end of the run)
        const int q = warp & 3;
        const int h = (warp - 2) >> 2;
        const int row = q * 32 + lane;  // packed filter row
        if (__all_sync(0xffffffffu, mbar_wait(acc_full, 0, abort_flag, a.status))) {
            tc_fence_after();
            float* dst = a.slices + ((size_t)blockIdx.x * a.bn + row) * a.cols;
            const int nch = a.cols / kEpiCols;  // cols is a multiple of 16
            for (int k = h; k < nch; k += 2) {
                uint32_t r[kEpiCols];
                tmem_ld_32x32b_x16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(k * kEpiCols), r);
                tmem_ld_wait();
                if (row < a.bn) {
                    float4* d4 = reinterpret_cast<float4*>(dst + k * kEpiCols);
#pragma unroll
                    for (int j = 0; j < kEpiCols / 4; ++j)
                        d4[j] = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                            __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, 512u);
    }
}

// dW[f_i][scol[j]] = sum over the CTAs' slices, in CTA order (deterministic).
__global__ void __launch_bounds__(256) k_wgrad_slab_reduce(const float* __restrict__ slices, int grid, int bn,
                                                           int cols, int kept, const int* __restrict__ rowmap,
                                                           const int* __restrict__ scol, int K, float* dW)
{
    pdl_wait();  // after the kernel before it in the stream
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const int i = blockIdx.y;
    if (j >= cols || i >= kept) return;
    const int col = __ldg(scol + j), f = __ldg(rowmap + i);
    if (col < 0 || f < 0) return;
    float acc = 0.0f;
    for (int b = 0; b < grid; ++b) acc += __ldg(slices + ((size_t)b * bn + i) * cols + j);
    dW[(size_t)f * K + col] = acc;
}

int wg_stage_stride(const sadmm_plan* plan)
{
    return (int)round_up((long long)plan->xs_cs * plan->xs_sp * 2, 1024) + 2 * kWgDzBox;
}

}  // namespace

bool wgrad_slab_ok(const sadmm_plan* plan, const Geometry& g)
{
    if (!plan->xs_mode || g.groups != 1 || plan->bn > 128 || plan->n_tiles != 1) return false;
    const long long cols = (long long)plan->xs_r * plan->xs_q * plan->xs_cs;
    if (cols > 512 || plan->xs_cs % 16 || plan->xs_cs > 64) return false;
    const long long room = kWgSmemLimit - 1024 - 256;
    return room / wg_stage_stride(plan) >= 2;
}

size_t wgrad_slab_bytes(const sadmm_plan* plan, const Geometry& g)
{
    if (!wgrad_slab_ok(plan, g)) return 0;
    const long long mt = (g.oh * plan->xs_wb + 127) / 128;
    const long long cols = (long long)plan->xs_r * plan->xs_q * plan->xs_cs;
    return (size_t)round_up(g.n * plan->bn * mt * 128 * 2, 1024) + (size_t)(kWgMaxCtas * plan->bn * cols * 4);
}

sadmm_status launch_wgrad_slab(const sadmm_plan* plan, const Geometry& g, const void* x, const void* dy,
                               const void* y, int ydt, int relu, float* dW, void* ws, cudaStream_t s)
{
    if (!wgrad_slab_ok(plan, g)) return SADMM_EINVAL;
    const char* base = static_cast<const char*>(plan->dev);
    const long long mt = (g.oh * plan->xs_wb + 127) / 128;
    const long long pg = mt * 128;
    const long long units = g.n * mt;
    if (units >= (1ll << 31) - (1ll << 20) || g.n * plan->bn >= (1ll << 31)) return SADMM_EUNSUPPORTED;
    // the forward's space-to-depth pass on this x, into the plan's copy
    sadmm_status st = launch_conv_slab(plan, g, x, nullptr, 0, nullptr, SADMM_FP32, SADMM_FWD_INPUT, s);
    if (st != SADMM_OK) return st;
    __nv_bfloat16* dzt = static_cast<__nv_bfloat16*>(ws);
    float* slices = reinterpret_cast<float*>(static_cast<char*>(ws) + round_up(g.n * plan->bn * pg * 2, 1024));
    const int* rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    const int* scol = reinterpret_cast<const int*>(base + plan->off_scol);
    const int kept = plan->n_filt;
    if (launch_pdl(k_slab_dzt, dim3((unsigned)((pg + 255) / 256), (unsigned)plan->bn, (unsigned)g.n), dim3(256), 0,
                   s, static_cast<const __nv_bfloat16*>(dy), y, ydt, relu, rowmap, kept, plan->bn, (int)g.f,
                   (int)g.oh, (int)g.ow, plan->xs_wb, (int)pg, dzt) != cudaSuccess)
        return SADMM_ECUDA;

    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return SADMM_ECUDA;
    alignas(64) CUtensorMap td;
    {
        // dZ [N*bn rows][pg pixels]: boxes of 64 pixels x 128 rows, 128-byte swizzle
        // (rows past an image's bn belong to the next image or read as zero: they
        // only feed accumulator rows no slice keeps)
        memset(&td, 0, sizeof(td));
        const cuuint64_t gdim[2] = {(cuuint64_t)pg, (cuuint64_t)(g.n * plan->bn)};
        const cuuint64_t gstride[1] = {(cuuint64_t)pg * 2};
        const cuuint32_t box[2] = {64u, 128u};
        const cuuint32_t estride[2] = {1u, 1u};
        if (enc(&td, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, dzt, gdim, gstride, box, estride,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return SADMM_ECUDA;
    }
    CUtensorMap tx;
    memcpy(&tx, plan->tmap_xs, sizeof(tx));

    WgArgs a;
    memset(&a, 0, sizeof(a));
    a.units = (int)units;
    a.MT = (int)mt;
    a.mt_div = make_fastdiv((uint32_t)mt);
    a.sp = plan->xs_sp;
    a.R = plan->xs_r;
    a.Q = plan->xs_q;
    a.Wb = plan->xs_wb;
    a.cs = plan->xs_cs;
    a.nchunks = plan->xs_cs / 8;
    a.bn = plan->bn;
    a.cols = plan->xs_r * plan->xs_q * plan->xs_cs;
    a.stage_stride = wg_stage_stride(plan);
    a.slab_bytes = plan->xs_cs * plan->xs_sp * 2;
    long long stages = (kWgSmemLimit - 1024 - 256) / a.stage_stride;
    if (stages > kWgMaxStages) stages = kWgMaxStages;
    a.stages = (int)stages;
    a.slices = slices;
    a.status = device_status_ptr();
    long long grid = std::min<long long>(std::min<long long>(device_sm_count(), kWgMaxCtas), units);
    const size_t smem = 1024 + (size_t)a.stages * a.stage_stride + 256;
    static int configured_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_dev != dev) {
        if (cudaFuncSetAttribute(k_wgrad_slab, cudaFuncAttributeMaxDynamicSharedMemorySize, kWgSmemLimit) !=
            cudaSuccess)
            return SADMM_ECUDA;
        configured_dev = dev;
    }
    if (launch_pdl(k_wgrad_slab, dim3((unsigned)grid), dim3(kWgThreads), smem, s, tx, td, a) != cudaSuccess)
        return SADMM_ECUDA;
    if (launch_pdl(k_wgrad_slab_reduce, dim3((unsigned)((a.cols + 255) / 256), (unsigned)kept), dim3(256), 0, s,
                   static_cast<const float*>(slices), (int)grid, a.bn, a.cols, kept, rowmap, scol, (int)g.k,
                   dW) != cudaSuccess)
        return SADMM_ECUDA;
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
