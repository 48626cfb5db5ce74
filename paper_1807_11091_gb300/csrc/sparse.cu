// sparse.cu -- CONV forward over a non-structured (element-wise) sparse weight
// tensor, the comparison point of the paper's speed tests (Sec. 5: weights
// pruned element by element, run through a sparse library, speed up little or
// slow down on a GPU, where structured pruning gives a smaller dense GEMM).
//
//   k_sparse_count  one block per filter: kept entries of the filter's row
//   k_sparse_scan   one block: row pointers = exclusive prefix sum of the counts
//   k_sparse_fill   one block per filter: the row's kept entries in column
//                   order, each {x offset of the column, tap bits, weight}
//   k_sparse_conv   one thread per output pixel and a block per (pixel tile,
//                   filter): y = ReLU(bias + sum over the filter's kept entries
//                   of w * x), fp32 on the CUDA cores (a sparse matrix has no
//                   dense tile for the tensor cores to take)
//
// Plan buffer (caller-owned): row pointers [F + 1] int32 (rounded up to 256 B),
// then entries [capacity] of 16 bytes.
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kSparseThreads = 256;

struct SparseGeom {
    int F, K, taps, KH, KW, split;
    long long thw;
    int hw, W;
};

// x offset (relative to the pixel's window origin) and tap bits of GEMM column j.
SADMM_DEV int4 column_entry(const SparseGeom& s, int j, float w)
{
    const int c = j / s.taps, r = j - c * s.taps;
    const int kt = r / (s.KH * s.KW), kh = (r / s.KW) % s.KH, kw = r % s.KW;
    int4 e;
    e.x = (int)((long long)c * s.thw + (long long)kt * s.hw + kh * s.W + kw);
    e.y = s.split ? (int)((1u << (kt * s.KH + kh)) | (1u << (16 + kw))) : (int)(1u << r);
    e.z = __float_as_int(w);
    e.w = 0;
    return e;
}

__global__ void __launch_bounds__(kSparseThreads) k_sparse_count(const uint8_t* keep, int K, int* row_ptr)
{
    pdl_wait();
    const int f = blockIdx.x;
    const uint8_t* row = keep + (long long)f * K;
    int n = 0;
    for (int j = threadIdx.x; j < K; j += blockDim.x) n += row[j] != 0;
    for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
    __shared__ int s_part[kSparseThreads / 32];
    if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = n;
    __syncthreads();
    if (threadIdx.x == 0) {
        int t = 0;
        for (int w = 0; w < kSparseThreads / 32; ++w) t += s_part[w];
        row_ptr[f + 1] = t;  // the scan turns counts into pointers in place
    }
}

// Exclusive scan of row_ptr[1..F] (the counts) in place, row_ptr[0] = 0.  When
// the total exceeds the plan's capacity, every row is emptied and the status
// word raised.
__global__ void __launch_bounds__(1024) k_sparse_scan(int* row_ptr, int F, long long capacity, int* status)
{
    pdl_wait();
    __shared__ int s_warp[32];
    __shared__ long long s_carry;
    if (threadIdx.x == 0) s_carry = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int base = 0; base < F; base += blockDim.x) {
        const int i = base + threadIdx.x;
        const int v = i < F ? row_ptr[i + 1] : 0;
        int incl = v;
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += u;
        }
        if (lane == 31) s_warp[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int w = lane < (int)(blockDim.x >> 5) ? s_warp[lane] : 0;
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += u;
            }
            s_warp[lane] = w;  // inclusive sums of the warps
        }
        __syncthreads();
        const long long before = s_carry + (warp > 0 ? s_warp[warp - 1] : 0);
        if (i < F) row_ptr[i + 1] = (int)min(before + incl, (long long)0x7fffffff);
        __syncthreads();
        if (threadIdx.x == 0) s_carry += s_warp[(blockDim.x >> 5) - 1];
        __syncthreads();
    }
    if (threadIdx.x == 0) row_ptr[0] = 0;
    if (s_carry > capacity) {
        if (threadIdx.x == 0) raise_status(status, kDevBadIndex);
        __syncthreads();
        for (int i = threadIdx.x; i <= F; i += blockDim.x) row_ptr[i] = 0;
    }
}

// Entries of filter f in column order: a block-wide ordered compaction of the
// row's keep flags, chunk by chunk.
template <typename T>
__global__ void __launch_bounds__(kSparseThreads)
    k_sparse_fill(const T* W, const uint8_t* keep, SparseGeom s, const int* row_ptr, int4* entries)
{
    pdl_wait();
    const int f = blockIdx.x;
    const long long row0 = (long long)f * s.K;
    int out = row_ptr[f];
    const int end = row_ptr[f + 1];
    __shared__ int s_warp[kSparseThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int base = 0; base < s.K && out < end; base += kSparseThreads) {
        const int j = base + threadIdx.x;
        const bool k = j < s.K && keep[row0 + j] != 0;
        const unsigned bal = __ballot_sync(0xffffffffu, k);
        if (lane == 0) s_warp[warp] = __popc(bal);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < kSparseThreads / 32; ++w) {
            if (w < warp) before += s_warp[w];
            total += s_warp[w];
        }
        const int pos = out + before + __popc(bal & ((1u << lane) - 1u));
        if (k && pos < end) entries[pos] = column_entry(s, j, static_cast<float>(W[row0 + j]));
        out += total;
        __syncthreads();
    }
}

struct SparseConvArgs {
    const unsigned short* x;
    const float* bias;
    const int* row_ptr;
    const int4* entries;
    void* y;
    int M, plane, OHW, OW, F, Cg, Fg;
    int T, H, W, KT, KH, KW, st, sh, sw, pt, ph, pw, split;
    long long x_chw, thw;
    int hw, relu;
    long long x_total, y_total;  // elements of x and y (the debug build's index checks)
    int* status;
};

template <bool OUT_BF16>
__global__ void __launch_bounds__(kSparseThreads) k_sparse_conv(const SparseConvArgs a)
{
    pdl_wait();
    const int f = blockIdx.y;
    const int m = blockIdx.x * kSparseThreads + threadIdx.x;
    if (m >= a.M) return;
    const int n = m / a.plane, pix = m - n * a.plane;
    const int ot = pix / a.OHW, r2 = pix - ot * a.OHW;
    const int oh = r2 / a.OW, ow = r2 - oh * a.OW;
    const int it0 = ot * a.st - a.pt, ih0 = oh * a.sh - a.ph, iw0 = ow * a.sw - a.pw;
    const uint32_t M = tap_mask(it0, ih0, iw0, a.KT, a.KH, a.KW, a.T, a.H, a.W, a.split);
    const int g = f / a.Fg;
    const unsigned short* xb =
        a.x + ((long long)n * a.x_chw + (long long)g * a.Cg * a.thw + (long long)it0 * a.hw + (long long)ih0 * a.W + iw0);
    const int e0 = __ldg(a.row_ptr + f), e1 = __ldg(a.row_ptr + f + 1);
    float acc = 0.0f;
    for (int e = e0; e < e1; ++e) {
        const int4 t = __ldg(a.entries + e);
        const uint32_t bits = (uint32_t)t.y;
        if ((M & bits) == bits && dbg_in(xb + t.x - a.x, a.x_total, a.status)) {
            const float xv = __uint_as_float((uint32_t)__ldg(xb + t.x) << 16);
            acc = fmaf(__int_as_float(t.z), xv, acc);
        }
    }
    float v = acc + (a.bias ? __ldg(a.bias + f) : 0.0f);
    if (a.relu) v = fmaxf(v, 0.0f);
    const long long off = ((long long)n * a.F + f) * a.plane + pix;
    if (!dbg_in(off, a.y_total, a.status)) return;
    if (OUT_BF16)
        reinterpret_cast<__nv_bfloat16*>(a.y)[off] = __float2bfloat16_rn(v);
    else
        reinterpret_cast<float*>(a.y)[off] = v;
}

SparseGeom sparse_geom(const Geometry& g)
{
    SparseGeom s;
    s.F = (int)g.f;
    s.K = (int)g.k;
    s.taps = (int)g.taps;
    s.KH = (int)g.kh;
    s.KW = (int)g.kw;
    s.split = tap_mask_mode(g);
    s.thw = g.t * g.h * g.w;
    s.hw = (int)(g.h * g.w);
    s.W = (int)g.w;
    return s;
}

}  // namespace

size_t sparse_plan_bytes(const Geometry& g, long long capacity)
{
    return (size_t)round_up((g.f + 1) * 4, 256) + (size_t)capacity * 16;
}

sadmm_status launch_sparse_pack(const Geometry& g, const void* W, int wdt, const uint8_t* keep, void* buf,
                                long long capacity, cudaStream_t s)
{
    int* row_ptr = static_cast<int*>(buf);
    int4* entries = reinterpret_cast<int4*>(static_cast<char*>(buf) + round_up((g.f + 1) * 4, 256));
    const SparseGeom sg = sparse_geom(g);
    cudaError_t e = launch_pdl(k_sparse_count, dim3((unsigned)g.f), dim3(kSparseThreads), 0, s, keep, sg.K, row_ptr);
    if (e == cudaSuccess)
        e = launch_pdl(k_sparse_scan, dim3(1), dim3(1024), 0, s, row_ptr, sg.F, capacity, device_status_ptr());
    if (e == cudaSuccess) {
        if (wdt == SADMM_BF16)
            e = launch_pdl(k_sparse_fill<__nv_bfloat16>, dim3((unsigned)g.f), dim3(kSparseThreads), 0, s,
                           static_cast<const __nv_bfloat16*>(W), keep, sg, (const int*)row_ptr, entries);
        else
            e = launch_pdl(k_sparse_fill<float>, dim3((unsigned)g.f), dim3(kSparseThreads), 0, s,
                           static_cast<const float*>(W), keep, sg, (const int*)row_ptr, entries);
    }
    return e == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

sadmm_status launch_sparse_conv(const Geometry& g, const void* buf, const void* x, const float* bias, int relu,
                                void* y, int ydt, cudaStream_t s)
{
    SparseConvArgs a;
    memset(&a, 0, sizeof(a));
    a.x = static_cast<const unsigned short*>(x);
    a.bias = bias;
    a.row_ptr = static_cast<const int*>(buf);
    a.entries = reinterpret_cast<const int4*>(static_cast<const char*>(buf) + round_up((g.f + 1) * 4, 256));
    a.y = y;
    if (g.m >= (1ll << 31) - kSparseThreads) return SADMM_EUNSUPPORTED;
    a.M = (int)g.m;
    a.plane = (int)g.plane;
    a.OHW = (int)(g.oh * g.ow);
    a.OW = (int)g.ow;
    a.F = (int)g.f;
    a.Cg = (int)g.cg;
    a.Fg = (int)g.fg;
    a.T = (int)g.t;
    a.H = (int)g.h;
    a.W = (int)g.w;
    a.KT = (int)g.kt;
    a.KH = (int)g.kh;
    a.KW = (int)g.kw;
    a.st = (int)g.st;
    a.sh = (int)g.sh;
    a.sw = (int)g.sw;
    a.pt = (int)g.pt;
    a.ph = (int)g.ph;
    a.pw = (int)g.pw;
    a.split = tap_mask_mode(g);
    a.x_chw = g.c * g.t * g.h * g.w;
    a.thw = g.t * g.h * g.w;
    a.hw = (int)(g.h * g.w);
    a.x_total = g.n * g.c * g.t * g.h * g.w;
    a.y_total = g.n * g.f * g.plane;
    a.status = device_status_ptr();
    a.relu = relu ? 1 : 0;
    if (g.f > 65535) return SADMM_EUNSUPPORTED;
    const dim3 grid((unsigned)((g.m + kSparseThreads - 1) / kSparseThreads), (unsigned)g.f);
    const cudaError_t e =
        (ydt == SADMM_BF16) ? launch_pdl(k_sparse_conv<true>, grid, dim3(kSparseThreads), 0, s, a)
                            : launch_pdl(k_sparse_conv<false>, grid, dim3(kSparseThreads), 0, s, a);
    return e == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
