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
//   k_admm_apply  one pass over the [F][K] matrices of every layer of the
//                 batch: read W and U, write Z and U^{k+1}.  HBM bound: 2
//                 reads + 2 writes per element.
#include <string.h>

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

// Per-layer parameters of the batched apply pass.
struct ApplyLayer {
    const void* W;
    void* U;
    void* Z;
    const uint8_t* rkeep;
    const uint8_t* ckeep;  // NULL: every column kept
    int K, cblocks;        // cblocks: 1024-column blocks per row
    uint32_t tmul, tshift; // group of column j: (umulhi(j, tmul) + j) >> tshift
    long long b0;          // first block of this layer
};

struct ApplyArgs {
    int n;
    ApplyLayer L[kMaxBatch];
};

// Block b of the batch: row a and columns bx*1024 .. bx*1024+1023 of its
// layer, kApplyCols per thread at a stride of kApplyThreads (coalesced).
// Column j keeps when its group's flag is set: ckeep[j] (shape-wise),
// ckeep[j / taps] (channel-wise), always (ckeep == NULL).  The division by
// taps is q = (umulhi(j, tmul) + j) >> tshift (exact for j < 2^31).
template <typename T>
__global__ void __launch_bounds__(kApplyThreads) k_admm_apply(const __grid_constant__ ApplyArgs aa)
{
    pdl_wait();  // after the kernel before it in the stream
    const long long b = blockIdx.x;
    int l = 0, hi = aa.n - 1;
    while (l < hi) {
        const int mid = (l + hi + 1) >> 1;
        if (aa.L[mid].b0 <= b) l = mid;
        else hi = mid - 1;
    }
    const ApplyLayer& L = aa.L[l];
    const int local = (int)(b - L.b0);
    const int a = local / L.cblocks, bx = local - a * L.cblocks;
    const T* __restrict__ W = static_cast<const T*>(L.W);
    T* __restrict__ U = static_cast<T*>(L.U);
    T* __restrict__ Z = static_cast<T*>(L.Z);
    const int K = L.K;
    const bool rk = L.rkeep[a] != 0;
    const long long base = (long long)a * K;
    const int j0 = bx * (kApplyThreads * kApplyCols) + threadIdx.x;
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
            const uint32_t grp = (__umulhi((uint32_t)j, L.tmul) + (uint32_t)j) >> L.tshift;
            const bool keep = rk && (!L.ckeep || L.ckeep[grp] != 0);
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

sadmm_status launch_admm_batch(const ProjItem* items, int n, int wdt, cudaStream_t s)
{
    if (n < 1 || n > kMaxBatch) return SADMM_EINVAL;
    ProjItem pit[kMaxBatch];
    ApplyArgs aa;
    memset(&aa, 0, sizeof(aa));
    aa.n = n;
    long long blocks = 0;
    for (int l = 0; l < n; ++l) {
        const Geometry& g = items[l].g;
        pit[l] = items[l];
        // keep flags after the projection's scratch in the item's workspace
        uint8_t* rkeep =
            static_cast<uint8_t*>(items[l].ws) + round_up((long long)project_workspace_bytes(g, items[l].colkind), 256);
        uint8_t* ckeep = rkeep + round_up(g.f, 256);
        pit[l].rkeep = rkeep;
        pit[l].ckeep = items[l].colkind == SADMM_COL_NONE ? nullptr : ckeep;
        ApplyLayer& L = aa.L[l];
        L.W = items[l].W;
        L.U = const_cast<void*>(items[l].U);
        L.Z = items[l].Z;
        L.rkeep = rkeep;
        L.ckeep = pit[l].ckeep;
        L.K = (int)g.k;
        L.cblocks = (int)((g.k + kApplyThreads * kApplyCols - 1) / (kApplyThreads * kApplyCols));
        // group of column j: j (shape), j / taps (channel); multiply-shift constants
        const uint32_t d = (items[l].colkind == SADMM_COL_CHANNEL) ? (uint32_t)g.taps : 1u;
        uint32_t sh = 0;
        while ((1ull << sh) < d) ++sh;
        L.tmul = (uint32_t)((((1ull << sh) - d) << 32) / d + 1);
        L.tshift = sh;
        L.b0 = blocks;
        blocks += (long long)g.f * L.cblocks;
    }
    if (blocks >= (1ll << 31)) return SADMM_EUNSUPPORTED;
    sadmm_status st = launch_project_batch(pit, n, wdt, s);
    if (st != SADMM_OK) return st;
    if (wdt == SADMM_BF16)
        launch_pdl(k_admm_apply<__nv_bfloat16>, dim3((unsigned)blocks), dim3(kApplyThreads), 0, s, aa);
    else
        launch_pdl(k_admm_apply<float>, dim3((unsigned)blocks), dim3(kApplyThreads), 0, s, aa);
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

sadmm_status launch_admm_update(const Geometry& g, const void* W, void* U, void* Z, int wdt, int k_filters,
                                int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out, void* ws,
                                cudaStream_t s)
{
    ProjItem it;
    it.g = g;
    it.W = W;
    it.U = U;
    it.Z = Z;
    it.k_filters = k_filters;
    it.colkind = colkind;
    it.k_cols = k_cols;
    it.filt_idx = filt_idx;
    it.col_idx = col_idx;
    it.keys_out = keys_out;
    it.ws = ws;
    it.rkeep = nullptr;
    it.ckeep = nullptr;
    return launch_admm_batch(&it, 1, wdt, s);
}

}  // namespace sadmm
