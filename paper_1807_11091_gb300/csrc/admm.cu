// admm.cu -- the ADMM Z- and U-update of one layer (Sec. 4).
//
// The Z-subproblem's optimum is the Euclidean projection of
// V = W^{k+1} + U^k onto the structured-sparsity set S (Eq. 4 and the
// filter-/channel-/shape-wise solutions of Sec. 4), and the scaled dual then
// moves to U^{k+1} = U^k + W^{k+1} - Z^{k+1}.  With V formed once in the
// tensors' precision, Z keeps V on the kept groups and is zero elsewhere, and
// U^{k+1} = V - Z is zero on the kept groups and V elsewhere.
//
// After the projection kernels of project.cu have selected the kept filters
// and column groups from V (and written a keep flag per group),
//   k_admm_apply  one pass over the [F][K] matrix: read W and U, write Z and
//                 U^{k+1}.  HBM bound: 2 reads + 2 writes per element.
#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kApplyThreads = 256;
constexpr int kApplyCols = 4;  // columns per thread

// V = W + U rounded once to the tensors' type (fp32 add; bf16 inputs add
// exactly in fp32 unless their exponents differ by more than 16, and the
// result is then rounded to nearest even).
SADMM_DEV float vsum(float w, float u) { return w + u; }
SADMM_DEV __nv_bfloat16 vsum(__nv_bfloat16 w, __nv_bfloat16 u)
{
    return __float2bfloat16_rn(__bfloat162float(w) + __bfloat162float(u));
}
template <typename T>
SADMM_DEV T zero_of();
template <>
SADMM_DEV float zero_of<float>() { return 0.0f; }
template <>
SADMM_DEV __nv_bfloat16 zero_of<__nv_bfloat16>() { return __float2bfloat16_rn(0.0f); }

// Block (bx, a): row a, columns bx*1024 .. bx*1024+1023, kApplyCols per thread
// at a stride of kApplyThreads (coalesced).
// Column j keeps when its group's flag is set: ckeep[j] (shape-wise),
// ckeep[j / taps] (channel-wise), always (ckeep == NULL).  The division by
// taps is q = (umulhi(j, tmul) + j) >> tshift (exact for j < 2^31).
template <typename T>
__global__ void __launch_bounds__(kApplyThreads) k_admm_apply(const T* __restrict__ W, T* __restrict__ U,
                                                              T* __restrict__ Z, int K,
                                                              const uint8_t* __restrict__ rkeep,
                                                              const uint8_t* __restrict__ ckeep, uint32_t tmul,
                                                              uint32_t tshift)
{
    pdl_wait();  // after the kernel before it in the stream
    const int a = blockIdx.y;
    const bool rk = rkeep[a] != 0;
    const long long base = (long long)a * K;
    const int j0 = blockIdx.x * (kApplyThreads * kApplyCols) + threadIdx.x;
    T w[kApplyCols], u[kApplyCols];
#pragma unroll
    for (int q = 0; q < kApplyCols; ++q) {
        const int j = j0 + q * kApplyThreads;
        if (j < K) {
            w[q] = W[base + j];
            u[q] = U[base + j];
        }
    }
#pragma unroll
    for (int q = 0; q < kApplyCols; ++q) {
        const int j = j0 + q * kApplyThreads;
        if (j < K) {
            const T v = vsum(w[q], u[q]);
            const uint32_t grp = (__umulhi((uint32_t)j, tmul) + (uint32_t)j) >> tshift;
            const bool keep = rk && (!ckeep || ckeep[grp] != 0);
            Z[base + j] = keep ? v : zero_of<T>();
            U[base + j] = keep ? zero_of<T>() : v;
        }
    }
}

size_t mask_bytes(const Geometry& g) { return (size_t)(round_up(g.f, 256) + round_up(g.k, 256)); }

}  // namespace

size_t admm_workspace_bytes(const Geometry& g, int colkind)
{
    return round_up((long long)project_workspace_bytes(g, colkind), 256) + mask_bytes(g);
}

sadmm_status launch_admm_update(const Geometry& g, const void* W, void* U, void* Z, int wdt, int k_filters,
                                int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out, void* ws,
                                cudaStream_t s)
{
    uint8_t* rkeep = static_cast<uint8_t*>(ws) + round_up((long long)project_workspace_bytes(g, colkind), 256);
    uint8_t* ckeep = rkeep + round_up(g.f, 256);
    sadmm_status st = launch_project(g, W, U, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out, ws, s,
                                     rkeep, colkind == SADMM_COL_NONE ? nullptr : ckeep);
    if (st != SADMM_OK) return st;
    const int F = (int)g.f, K = (int)g.k;
    // group of column j: j (shape), j / taps (channel); multiply-shift constants
    const uint32_t d = (colkind == SADMM_COL_CHANNEL) ? (uint32_t)g.taps : 1u;
    uint32_t sh = 0;
    while ((1ull << sh) < d) ++sh;
    const uint32_t mul = (uint32_t)((((1ull << sh) - d) << 32) / d + 1);
    const uint8_t* ck = (colkind == SADMM_COL_NONE) ? nullptr : ckeep;
    const dim3 grid((unsigned)((K + kApplyThreads * kApplyCols - 1) / (kApplyThreads * kApplyCols)), (unsigned)F);
    if (wdt == SADMM_BF16)
        launch_pdl(k_admm_apply<__nv_bfloat16>, grid, dim3(kApplyThreads), 0, s,
                   static_cast<const __nv_bfloat16*>(W), static_cast<__nv_bfloat16*>(U),
                   static_cast<__nv_bfloat16*>(Z), K, static_cast<const uint8_t*>(rkeep), ck, mul, sh);
    else
        launch_pdl(k_admm_apply<float>, grid, dim3(kApplyThreads), 0, s, static_cast<const float*>(W),
                   static_cast<float*>(U), static_cast<float*>(Z), K, static_cast<const uint8_t*>(rkeep), ck, mul,
                   sh);
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
