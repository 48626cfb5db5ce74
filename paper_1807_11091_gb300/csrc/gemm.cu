// gemm.cu -- a plain bf16 GEMM on the sm_103a tensor cores, used by the
// masked-retraining backward (bwd.cu): C = A * B^T with A [M][K] and B [N][K]
// (both K-contiguous), fp32 accumulation in TMEM, optional accumulation into
// C.  One CTA per 128 x bn tile of C:
//   warp 0      TMA producer: 64-column boxes of A (128 rows) and B (bn rows),
//               128-byte swizzle, up to 4 stages in flight
//   warp 1      TMEM allocator and the single thread issuing
//               tcgen05.mma.cta_group::1.kind::f16 (M = 128, N = bn, K = 16)
//   warps 2-5   epilogue: tcgen05.ld of the accumulator (lane = row of C),
//               16-byte stores (adding the previous C when accumulating)
#include <cuda.h>
#include <cudaTypedefs.h>
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace sadmm {

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn();  // pack.cu

namespace {

constexpr int kGemmThreads = 192;
constexpr int kGemmStages = 4;
constexpr int kATile = 128 * 128;  // 128 rows x 64 bf16

struct GemmArgs {
    float* C;
    long long ldc;
    int nk;  // K / 64 stages of this CTA (its split)
    int bn;
    int accumulate;  // 0: C = product; 1: C += product; 2: C += product with atomics (split K)
    long long slice;  // > 0: split z owns C + z * slice (its own slice, no atomics)
    int tmem_cols;
    int* status;
};

__global__ void __launch_bounds__(kGemmThreads, 1)
    k_gemm(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb, const GemmArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t b_bytes = (uint32_t)a.bn * 128u;
    uint8_t* sA = smem;
    uint8_t* sB = smem + kGemmStages * kATile;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sB + (size_t)kGemmStages * b_bytes);
    uint64_t* full = bars;
    uint64_t* empty = bars + kGemmStages;
    uint64_t* acc_full = bars + 2 * kGemmStages;
    uint64_t* drain = acc_full + 1;
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * 128, n0 = blockIdx.y * a.bn;
    const int k0 = blockIdx.z * a.nk * 64;  // first K column of this split

    if (threadIdx.x == 0) {
        for (int s = 0; s < kGemmStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(acc_full, 1);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, (uint32_t)a.tmem_cols);
        tmem_relinquish();
    }
    pdl_wait();  // nothing above reads global memory
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_desc(&ta);
            tma_prefetch_desc(&tb);
            int issued = 0;
            for (int ks = 0; ks < a.nk; ++ks) {
                const int s = ks % kGemmStages;
                const uint32_t ph = (uint32_t)(ks / kGemmStages) & 1u;
                if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) break;
                mbar_arrive_expect_tx(&full[s], (uint32_t)kATile + b_bytes);
                tma_load_2d(sA + (size_t)s * kATile, &ta, &full[s], k0 + ks * 64, m0);
                tma_load_2d(sB + (size_t)s * b_bytes, &tb, &full[s], k0 + ks * 64, n0);
                ++issued;
            }
            // the loads issued have landed before the CTA retires
            for (int q = (issued > kGemmStages ? issued - kGemmStages : 0); q < issued; ++q) {
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full[q % kGemmStages], (uint32_t)(q / kGemmStages) & 1u) &&
                       globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // the whole warp runs the loop; one elected lane issues the MMAs and commits
        {
            const uint32_t idesc = idesc_bf16_f32(128, a.bn);
            bool ok = true;
            for (int ks = 0; ks < a.nk; ++ks) {
                const int s = ks % kGemmStages;
                const uint32_t ph = (uint32_t)(ks / kGemmStages) & 1u;
                if (!mbar_wait_warp(&full[s], ph, abort_flag, a.status)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA + (size_t)s * kATile);
                const uint32_t b0 = smem_u32(sB + (size_t)s * b_bytes);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_bf16_ss_elect(tmem_base, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32), idesc,
                                (ks | kk) != 0 ? 1u : 0u);
                mma_commit_elect(&empty[s]);
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
        // epilogue: warp w reads TMEM lanes 32*(w%4) .. +31 = rows of C
        const int q = warp & 3;
        const int row = m0 + q * 32 + lane;
        if (__all_sync(0xffffffffu, mbar_wait(acc_full, 0, abort_flag, a.status))) {
            tc_fence_after();
            float* crow = a.C + (size_t)blockIdx.z * (size_t)a.slice + (size_t)row * a.ldc + n0;
            // 16-column chunks: bn is a multiple of 16, so no chunk passes the tile
            for (int c0 = 0; c0 < a.bn; c0 += 16) {
                uint32_t r[16];
                tmem_ld_32x32b_x16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, r);
                tmem_ld_wait();
                if (a.accumulate == 2) {
                    // split K: several CTAs add into the same tile
#pragma unroll
                    for (int j = 0; j < 16; ++j) atomicAdd(crow + c0 + j, __uint_as_float(r[j]));
                    continue;
                }
                float4* dst = reinterpret_cast<float4*>(crow + c0);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    float4 v = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                           __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
                    if (a.accumulate) {
                        const float4 o = dst[j];
                        v.x += o.x; v.y += o.y; v.z += o.z; v.w += o.w;
                    }
                    dst[j] = v;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, (uint32_t)a.tmem_cols);
    }
}

bool encode_kmajor(CUtensorMap* map, const void* base, long long rows, long long K, int box_rows)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return false;
    memset(map, 0, sizeof(*map));
    const cuuint64_t gdim[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    const cuuint64_t gstride[1] = {(cuuint64_t)K * 2};
    const cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
    const cuuint32_t estride[2] = {1u, 1u};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride, box, estride,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

sadmm_status launch_gemm(const void* A, const void* B, float* C, long long M, long long N, long long K,
                         long long ldc, int bn, bool accumulate, cudaStream_t s, int splits, long long slice)
{
    if (M <= 0 || N <= 0 || K <= 0) return SADMM_OK;
    if (M % 128 || bn < 16 || bn > 256 || bn % 16 || N % bn || K % 64 || ldc % 4 || ldc < N) return SADMM_EINVAL;
    if (splits < 1 || (K / 64) % splits != 0 || splits > 65535) return SADMM_EINVAL;
    if (M / 128 > 65535 * 1024ll || N / bn > 65535) return SADMM_EUNSUPPORTED;
    alignas(64) CUtensorMap ta, tb;
    if (!encode_kmajor(&ta, A, M, K, 128) || !encode_kmajor(&tb, B, N, K, bn)) return SADMM_ECUDA;
    GemmArgs a;
    a.C = C;
    a.ldc = ldc;
    a.nk = (int)(K / 64 / splits);
    a.bn = bn;
    if (slice < 0 || (slice > 0 && slice < M * ldc)) return SADMM_EINVAL;
    a.slice = splits > 1 ? slice : 0;
    a.accumulate = (splits > 1 && slice == 0) ? 2 : (accumulate ? 1 : 0);
    int cols = 32;
    while (cols < bn) cols <<= 1;
    a.tmem_cols = cols;
    a.status = device_status_ptr();
    const size_t smem = 1024 + (size_t)kGemmStages * (kATile + (size_t)bn * 128) + 256;
    static int configured_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_dev != dev) {
        if (cudaFuncSetAttribute(k_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448) != cudaSuccess)
            return SADMM_ECUDA;
        configured_dev = dev;
    }
    const dim3 grid((unsigned)(M / 128), (unsigned)(N / bn), (unsigned)splits);
    if (launch_pdl(k_gemm, grid, dim3(kGemmThreads), smem, s, ta, tb, a) != cudaSuccess) return SADMM_ECUDA;
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
