// pack.cu -- compaction of the kept rows and columns of the lowered GEMM matrix
// (Sec. 3, "Combination of structured sparsities": filter-wise sparsity is row
// pruning and channel-/shape-wise sparsity is column pruning; what remains is a
// smaller full matrix).
//
//   k_pack_meta  one block per layer: per conv group the kept and pruned
//                filter lists and counts, the kept-column list and the gather
//                table (channel offset of each kept column in x plus its tap
//                bits); it also zeroes the plan's stream-K arrival counters.
//   k_pack_wp    one block per packed row of every layer:
//                Wp[g][i][j] = bf16(W[f_i][col_j]), zero outside the kept
//                counts, 16-byte stores.
// A call packs a batch of layers (sadmm_pack_batch; sadmm_pack is the batch of
// one): two launches whatever the batch size.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

struct PackArgs {
    const int* filt_idx;  // kept filters, ascending (unused when all_kept)
    int all_kept;         // n_filt == F
    const int* col_idx;   // NULL: all columns
    int n_filt, colkind, n_colgroups, n_cols;
    int F, groups, Fg, K, taps, KT, KH, KW;
    long long thw;  // T*H*W
    int hw, W;
    int k_pad, n_pad;
    int mask_mode;
    uint2* gather;
    int2* stage_chan;  // [k_pad/64] first and last channel of each stage
    int* colidx;
    int* rowmap;
    int* zeromap;
    int* counts;
    // input-slab plans (scol != NULL): slab column map and kept channel list
    int* scol;   // [xs_kpad] slab column -> GEMM column (-1: zero)
    int* chan;   // [xs_cs] kept input channels (-1 past them)
    int C, xs_cs, xs_kpad, xs_r, xs_q, sh, sw;
    int* skcnt;         // stream-K arrival counters, zeroed here
    int sk_n;
    int lists_in_smem;  // 1: the filter and column lists are staged in shared memory
};

// The layers of one pack launch, in kernel parameter space.
template <int N>
struct PackBatch {
    PackArgs L[N];
};

// One layer's rows for k_pack_wp: blocks first .. first + rows + srows - 1.
struct WpLayer {
    const void* W;
    const int* rowmap;
    const int* colidx;
    const int* scol;
    __nv_bfloat16* wp;
    __nv_bfloat16* wps;
    long long rows, first;
    int K, k_pad, kpad_s;
};

template <int N>
struct WpBatch {
    WpLayer L[N];
    int n;
};

// First position p in the ascending list a[0..n) with a[p] >= v.
SADMM_DEV int lower_bound(const int* a, int n, int v)
{
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (a[mid] < v) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// Dynamic shared memory (when the host passes enough): the filter and column
// lists, so the binary searches below read shared memory, not HBM.
SADMM_DEV void pack_meta(PackArgs a, int* status)
{
    __shared__ int s_start[65];
    __shared__ int s_bad;
    extern __shared__ int s_lists[];
    const int tid = threadIdx.x;
    for (int i = tid; i < a.sk_n; i += blockDim.x) a.skcnt[i] = 0;
    if (a.lists_in_smem) {
        int* fl = s_lists;
        int* cl = s_lists + (a.all_kept ? 0 : a.n_filt);
        if (!a.all_kept)
            for (int i = tid; i < a.n_filt; i += blockDim.x) fl[i] = a.filt_idx[i];
        if (a.col_idx && a.colkind != SADMM_COL_NONE)
            for (int i = tid; i < a.n_colgroups; i += blockDim.x) cl[i] = a.col_idx[i];
        __syncthreads();
        if (!a.all_kept) a.filt_idx = fl;
        if (a.col_idx && a.colkind != SADMM_COL_NONE) a.col_idx = cl;
    }
    // Index lists must be strictly ascending and in range.  A list that is not
    // gives a plan with every filter pruned and every column dropped (an
    // all-zero output) and raises the device status word.
    if (tid == 0) s_bad = 0;
    __syncthreads();
    if (!a.all_kept) {
        for (int i = tid; i < a.n_filt; i += blockDim.x) {
            const int v = a.filt_idx[i];
            if (v < 0 || v >= a.F || (i + 1 < a.n_filt && a.filt_idx[i + 1] <= v)) s_bad = 1;
        }
    }
    if (a.col_idx && a.colkind != SADMM_COL_NONE) {
        const int lim = (a.colkind == SADMM_COL_CHANNEL) ? a.K / a.taps : a.K;
        for (int i = tid; i < a.n_colgroups; i += blockDim.x) {
            const int v = a.col_idx[i];
            if (v < 0 || v >= lim || (i + 1 < a.n_colgroups && a.col_idx[i + 1] <= v)) s_bad = 1;
        }
    }
    __syncthreads();
    if (s_bad) {
        if (tid == 0) raise_status(status, kDevBadIndex);
        for (int g = tid; g < a.groups; g += blockDim.x) {
            a.counts[2 * g] = 0;
            a.counts[2 * g + 1] = a.Fg;
        }
        for (int r = tid; r < a.groups * a.n_pad; r += blockDim.x) a.rowmap[r] = -1;
        for (int f = tid; f < a.F; f += blockDim.x) a.zeromap[f] = f;
        for (int j = tid; j < a.k_pad; j += blockDim.x) {
            a.colidx[j] = -1;
            a.gather[j] = make_uint2(0u, 1u << 31);
        }
        for (int st = tid; st < a.k_pad / 64; st += blockDim.x) a.stage_chan[st] = make_int2(0, -1);
        if (a.scol) {
            for (int j = tid; j < a.xs_kpad; j += blockDim.x) a.scol[j] = -1;
            for (int ci = tid; ci < a.xs_cs; ci += blockDim.x) a.chan[ci] = -1;
        }
        return;
    }
    // kept-filter range of each conv group in the ascending filter list
    for (int g = tid; g <= a.groups; g += blockDim.x)
        s_start[g] = a.all_kept ? g * a.Fg : lower_bound(a.filt_idx, a.n_filt, g * a.Fg);
    __syncthreads();
    for (int g = tid; g < a.groups; g += blockDim.x) {
        const int kept = s_start[g + 1] - s_start[g];
        a.counts[2 * g] = kept;
        a.counts[2 * g + 1] = a.Fg - kept;
    }
    // rows of the packed matrix -> output filter (or -1 for padding rows)
    for (int r = tid; r < a.groups * a.n_pad; r += blockDim.x) {
        const int g = r / a.n_pad, i = r % a.n_pad;
        const int kept = s_start[g + 1] - s_start[g];
        int f = -1;
        if (i < kept) f = a.all_kept ? g * a.Fg + i : a.filt_idx[s_start[g] + i];
        a.rowmap[r] = f;
    }
    // pruned filters of each group, ascending
    if (!a.all_kept) {
        for (int f = tid; f < a.F; f += blockDim.x) {
            const int pos = lower_bound(a.filt_idx, a.n_filt, f);
            const bool kept = pos < a.n_filt && a.filt_idx[pos] == f;
            if (!kept) {
                const int g = f / a.Fg;
                const int z = (f - g * a.Fg) - (pos - s_start[g]);
                a.zeromap[g * a.Fg + z] = f;
            }
        }
    }
    // kept GEMM columns and their gather entries
    for (int j = tid; j < a.k_pad; j += blockDim.x) {
        int col = -1;
        if (j < a.n_cols) {
            if (a.colkind == SADMM_COL_SHAPE) col = a.col_idx[j];
            else if (a.colkind == SADMM_COL_CHANNEL) col = a.col_idx[j / a.taps] * a.taps + j % a.taps;
            else col = j;
        }
        a.colidx[j] = col;
        uint2 e = make_uint2(0u, 1u << 31);  // padding column: never inside the input
        if (col >= 0) {
            const int c = col / a.taps, r = col % a.taps;
            const int kt = r / (a.KH * a.KW), kh = (r / a.KW) % a.KH, kw = r % a.KW;
            e.x = (uint32_t)(c * a.thw + (long long)kt * a.hw + kh * a.W + kw);
            if (a.mask_mode == 0)
                e.y = 1u << r;
            else
                e.y = (1u << (kt * a.KH + kh)) | (1u << (16 + kw));
        }
        a.gather[j] = e;
    }
    __syncthreads();
    // channel range (first, last kept column's channel) of every 64-column stage
    for (int st = tid; st < a.k_pad / 64; st += blockDim.x) {
        const int j0 = st * 64, j1 = min(j0 + 63, a.n_cols - 1);
        a.stage_chan[st] = (j1 < j0) ? make_int2(0, -1) : make_int2(a.colidx[j0] / a.taps, a.colidx[j1] / a.taps);
    }
    if (a.scol) {
        // Slab column order of the input-slab path: column j is block tap
        // (r, q) = (j / cs / Q, j / cs % Q) and slab channel cc = j % cs =
        // (ci * sh + a) * sw + b, i.e. kept channel ci at phase (a, b); it holds
        // GEMM column chan[ci] * taps + (r*sh + a) * KW + q*sw + b, or nothing
        // (-1) past the kernel, the kept channels or the slab width.
        const int nck = a.colkind == SADMM_COL_CHANNEL ? a.n_colgroups : a.C;
        for (int ci = tid; ci < a.xs_cs; ci += blockDim.x)
            a.chan[ci] = ci < nck ? (a.colkind == SADMM_COL_CHANNEL ? a.col_idx[ci] : ci) : -1;
        const int rq_cols = a.xs_r * a.xs_q * a.xs_cs;
        for (int j = tid; j < a.xs_kpad; j += blockDim.x) {
            int col = -1;
            const int tap = j / a.xs_cs, cc = j - tap * a.xs_cs;
            const int r = tap / a.xs_q, q = tap - r * a.xs_q;
            const int ci = cc / (a.sh * a.sw), pa = (cc / a.sw) % a.sh, pb = cc % a.sw;
            const int kh = r * a.sh + pa, kw = q * a.sw + pb;
            if (j < rq_cols && ci < nck && kh < a.KH && kw < a.KW) {
                const int ch = a.colkind == SADMM_COL_CHANNEL ? a.col_idx[ci] : ci;
                col = ch * a.taps + kh * a.KW + kw;
            }
            a.scol[j] = col;
        }
    }
}

// Block b packs the meta data of layer b of the batch.
template <int N>
__global__ void __launch_bounds__(1024) k_pack_meta(const __grid_constant__ PackBatch<N> pb, int* status)
{
    pdl_wait();  // after the kernel before it in the stream
    pack_meta(pb.L[blockIdx.x], status);
}

template <typename T>
SADMM_DEV float load_f32(const T* p);
template <>
SADMM_DEV float load_f32<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }
template <>
SADMM_DEV float load_f32<float>(const float* p) { return *p; }

// Row r of a layer: rows past `rows` pack the input-slab plan's weights, row
// r - rows of conv group 0 through the slab column map scol, into wps [bn][kpad_s].
template <typename T>
SADMM_DEV void pack_wp_row(const WpLayer& L, long long r)
{
    const T* W = static_cast<const T*>(L.W);
    const int* colidx = L.colidx;
    int k_pad = L.k_pad;
    __nv_bfloat16* wp = L.wp;
    if (r >= L.rows) {
        r -= L.rows;
        colidx = L.scol;
        k_pad = L.kpad_s;
        wp = L.wps;
    }
    const int f = L.rowmap[r];
    uint4* dst = reinterpret_cast<uint4*>(wp + r * k_pad);
    for (int j8 = threadIdx.x; j8 < k_pad / 8; j8 += blockDim.x) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int j0 = j8 * 8 + 2 * e;
            const int c0 = colidx[j0], c1 = colidx[j0 + 1];
            const float v0 = (f >= 0 && c0 >= 0) ? load_f32<T>(W + (long long)f * L.K + c0) : 0.0f;
            const float v1 = (f >= 0 && c1 >= 0) ? load_f32<T>(W + (long long)f * L.K + c1) : 0.0f;
            const __nv_bfloat162 p = __floats2bfloat162_rn(v0, v1);  // .x = v0 (low half)
            w[e] = *reinterpret_cast<const uint32_t*>(&p);
        }
        dst[j8] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// Block b packs one row of the layer whose block range holds b.
template <typename T, int N>
__global__ void __launch_bounds__(128) k_pack_wp(const __grid_constant__ WpBatch<N> wb)
{
    pdl_wait();  // after the kernel before it in the stream
    const long long b = blockIdx.x;
    int lo = 0, hi = wb.n - 1;
    while (lo < hi) {  // the last layer whose first block is <= b
        const int mid = (lo + hi + 1) >> 1;
        if (wb.L[mid].first <= b) lo = mid;
        else hi = mid - 1;
    }
    pack_wp_row<T>(wb.L[lo], b - wb.L[lo].first);
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return nullptr;
        fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

namespace {

// The kernel arguments of one layer's meta data (plan->dev bound).
PackArgs pack_args(const sadmm_plan* plan, const Geometry& g, const int* filt_idx, const int* col_idx)
{
    char* base = static_cast<char*>(plan->dev);
    PackArgs a;
    memset(&a, 0, sizeof(a));
    a.all_kept = (plan->n_filt == (int)g.f) ? 1 : 0;
    a.filt_idx = a.all_kept ? nullptr : filt_idx;
    a.col_idx = col_idx;
    a.n_filt = plan->n_filt;
    a.colkind = plan->colkind;
    a.n_colgroups = plan->n_colgroups;
    a.n_cols = plan->n_cols;
    a.F = (int)g.f;
    a.groups = (int)g.groups;
    a.Fg = (int)g.fg;
    a.K = (int)g.k;
    a.taps = (int)g.taps;
    a.KT = (int)g.kt;
    a.KH = (int)g.kh;
    a.KW = (int)g.kw;
    a.thw = g.t * g.h * g.w;
    a.hw = (int)(g.h * g.w);
    a.W = (int)g.w;
    a.k_pad = plan->k_pad;
    a.n_pad = plan->n_pad;
    a.mask_mode = tap_mask_mode(g);
    a.gather = reinterpret_cast<uint2*>(base + plan->off_gather);
    a.stage_chan = reinterpret_cast<int2*>(a.gather + plan->k_pad);
    a.colidx = reinterpret_cast<int*>(base + plan->off_colidx);
    a.rowmap = reinterpret_cast<int*>(base + plan->off_rowmap);
    a.zeromap = reinterpret_cast<int*>(base + plan->off_zeromap);
    a.counts = reinterpret_cast<int*>(base + plan->off_counts);
    a.C = (int)g.c;
    if (plan->xs_mode) {
        a.scol = reinterpret_cast<int*>(base + plan->off_scol);
        a.chan = a.scol + plan->xs_kpad;
        a.xs_cs = plan->xs_cs;
        a.xs_kpad = plan->xs_kpad;
        a.xs_r = plan->xs_r;
        a.xs_q = plan->xs_q;
        a.sh = (int)g.sh;
        a.sw = (int)g.sw;
    }
    if (plan->sk_len > 0) {
        a.skcnt = reinterpret_cast<int*>(base + plan->off_sk);
        a.sk_n = plan->sk_grid;
    }
    return a;
}

// Bytes of the filter and column lists k_pack_meta stages in shared memory.
size_t list_bytes(const PackArgs& a)
{
    return (size_t)((a.all_kept ? 0 : a.n_filt) + ((a.col_idx && a.colkind != SADMM_COL_NONE) ? a.n_colgroups : 0)) *
           4;
}

constexpr size_t kListSmemCap = 40 * 1024;

// TMA descriptor of Wp: [groups*n_pad rows][k_pad bf16], boxes of 64 x bn,
// 128-byte swizzle (the layout the tensor-core operand descriptor expects);
// then those of a slab plan.
sadmm_status encode_maps(sadmm_plan* plan, const Geometry& g)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return SADMM_ECUDA;
    __nv_bfloat16* wp = reinterpret_cast<__nv_bfloat16*>(static_cast<char*>(plan->dev) + plan->off_wp);
    const unsigned rows = (unsigned)(g.groups * plan->n_pad);
    alignas(64) CUtensorMap map;
    memset(&map, 0, sizeof(map));
    const cuuint64_t gdim[2] = {(cuuint64_t)plan->k_pad, (cuuint64_t)rows};
    const cuuint64_t gstride[1] = {(cuuint64_t)plan->k_pad * 2};
    const cuuint32_t box[2] = {64u, (cuuint32_t)plan->bn};
    const cuuint32_t estride[2] = {1u, 1u};
    const CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wp, gdim, gstride, box, estride,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return SADMM_ECUDA;
    static_assert(sizeof(CUtensorMap) == sizeof(plan->tmap), "tensor map size");
    memcpy(plan->tmap, &map, sizeof(map));
    if (plan->xs_mode) return launch_pack_slab(plan, g);
    return SADMM_OK;
}

template <int N>
sadmm_status launch_batch(const PackJob* jobs, int n, int wdt, cudaStream_t s)
{
    PackBatch<N> pb;
    WpBatch<N> wb;
    memset(&pb, 0, sizeof(pb));
    memset(&wb, 0, sizeof(wb));
    size_t smem = 0;
    for (int i = 0; i < n; ++i) {
        pb.L[i] = pack_args(jobs[i].plan, jobs[i].g, jobs[i].filt_idx, jobs[i].col_idx);
        const size_t lb = list_bytes(pb.L[i]);
        if (lb <= kListSmemCap && lb > smem) smem = lb;
    }
    for (int i = 0; i < n; ++i) pb.L[i].lists_in_smem = list_bytes(pb.L[i]) <= smem ? 1 : 0;
    if (launch_pdl(k_pack_meta<N>, dim3((unsigned)n), dim3(1024), smem, s, pb, device_status_ptr()) != cudaSuccess)
        return SADMM_ECUDA;
    long long blocks = 0;
    for (int i = 0; i < n; ++i) {
        const sadmm_plan* plan = jobs[i].plan;
        const Geometry& g = jobs[i].g;
        char* base = static_cast<char*>(plan->dev);
        WpLayer& L = wb.L[i];
        L.W = jobs[i].W;
        L.K = (int)g.k;
        L.rowmap = pb.L[i].rowmap;
        L.colidx = pb.L[i].colidx;
        L.k_pad = plan->k_pad;
        L.wp = reinterpret_cast<__nv_bfloat16*>(base + plan->off_wp);
        L.rows = g.groups * plan->n_pad;
        // a slab plan also packs its weights in slab column order, in the same launch
        L.scol = pb.L[i].scol;
        L.kpad_s = plan->xs_kpad;
        L.wps = plan->xs_mode ? reinterpret_cast<__nv_bfloat16*>(base + plan->off_wps) : nullptr;
        L.first = blocks;
        blocks += L.rows + (plan->xs_mode ? plan->bn : 0);
    }
    wb.n = n;
    if (blocks >= (1ll << 31)) return SADMM_EUNSUPPORTED;
    const cudaError_t e =
        (wdt == SADMM_BF16)
            ? launch_pdl(k_pack_wp<__nv_bfloat16, N>, dim3((unsigned)blocks), dim3(128), 0, s, wb)
            : launch_pdl(k_pack_wp<float, N>, dim3((unsigned)blocks), dim3(128), 0, s, wb);
    if (e != cudaSuccess || cudaGetLastError() != cudaSuccess) return SADMM_ECUDA;
    for (int i = 0; i < n; ++i) {
        const sadmm_status st = encode_maps(jobs[i].plan, jobs[i].g);
        if (st != SADMM_OK) return st;
    }
    return SADMM_OK;
}

}  // namespace

sadmm_status launch_pack_batch(const PackJob* jobs, int n, int wdt, cudaStream_t s)
{
    if (n < 1 || n > kMaxBatch) return SADMM_EINVAL;
    return n == 1 ? launch_batch<1>(jobs, n, wdt, s) : launch_batch<kMaxBatch>(jobs, n, wdt, s);
}

sadmm_status launch_pack_slab(sadmm_plan* plan, const Geometry& g)
{
    // the slab column map, kept channels and slab-ordered weights were written
    // by k_pack_meta and k_pack_wp; here only their TMA descriptors
    char* base = static_cast<char*>(plan->dev);
    __nv_bfloat16* wps = reinterpret_cast<__nv_bfloat16*>(base + plan->off_wps);
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return SADMM_ECUDA;
    {
        // slab-ordered weights: [bn][xs_kpad], boxes of 64 columns x bn rows, 128-byte swizzle
        alignas(64) CUtensorMap map;
        memset(&map, 0, sizeof(map));
        const cuuint64_t gdim[2] = {(cuuint64_t)plan->xs_kpad, (cuuint64_t)plan->bn};
        const cuuint64_t gstride[1] = {(cuuint64_t)plan->xs_kpad * 2};
        const cuuint32_t box[2] = {64u, (cuuint32_t)plan->bn};
        const cuuint32_t estride[2] = {1u, 1u};
        if (enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, wps, gdim, gstride, box, estride,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return SADMM_ECUDA;
        memcpy(plan->tmap_ws, &map, sizeof(map));
    }
    {
        // space-to-depth input [N][cs/8][pimg][8] viewed as [N][cs/8][pimg/8][64]:
        // a box is one tile's slab, every chunk, as [chunk][sp pixels][8]
        // (no swizzle: the operand descriptors address 16-byte rows directly)
        alignas(64) CUtensorMap map;
        memset(&map, 0, sizeof(map));
        const long long oct = plan->xs_pimg / 8, chunks = plan->xs_cs / 8;
        const cuuint64_t gdim[4] = {64u, (cuuint64_t)oct, (cuuint64_t)chunks, (cuuint64_t)g.n};
        const cuuint64_t gstride[3] = {128u, (cuuint64_t)oct * 128u, (cuuint64_t)(chunks * oct * 128)};
        const cuuint32_t box[4] = {64u, (cuuint32_t)(plan->xs_sp / 8), (cuuint32_t)chunks, 1u};
        const cuuint32_t estride[4] = {1u, 1u, 1u, 1u};
        if (enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, base + plan->off_xs, gdim, gstride, box, estride,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return SADMM_ECUDA;
        memcpy(plan->tmap_xs, &map, sizeof(map));
    }
    return SADMM_OK;
}

}  // namespace sadmm
