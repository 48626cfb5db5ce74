// bwd.cu -- backward of a packed pruned CONV layer for masked retraining
// (Sec. 4, "Masked mapping and retraining": after the final projection the
// zero weights stay masked and only the kept weights are trained).
//
// With the layer's kept filters f_i (packed rows i) and kept GEMM columns
// col_j (packed columns j), dZ = dY * [y > 0] (ReLU fused in the forward),
// and A[m][j] the kept-column im2col of x for output pixel m:
//   dWp[i][j] = sum_m dZ[m][f_i] * A[m][j]          (weight gradient, kept only)
//   dA[m][j]  = sum_i dZ[m][f_i] * Wp[i][j]         (then col2im into dx)
//   db[f_i]   = sum_m dZ[m][f_i]
// Per conv group and per chunk of output pixels the two contractions run on
// the tensor cores (gemm.cu) over bf16 operands gathered here; the weight
// gradient's few output tiles split each chunk's pixels over many CTAs that
// add into dWp with fp32 atomics, and dx receives the col2im sums with fp32
// atomics.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

struct BwdGeo {
    const __nv_bfloat16* x;
    const __nv_bfloat16* dy;
    const void* y;
    int ydt, relu;
    const int* rowmap;   // [groups][n_pad] packed row -> filter (-1: padding)
    const int* colidx;   // [k_pad] packed column -> GEMM column (-1: padding)
    const int* counts;   // [groups][2] kept / pruned filters
    int N, C, T, H, W, F, Cg, Fg, groups;
    int KT, KH, KW, st, sh, sw, pt, ph, pw;
    int OT, OH, OW, plane, taps;
    long long M;  // N * plane
    int n_pad, k_pad, n_cols;
    int fr;       // filter rows of the wgrad operand: n_pad rounded up to 128
    int fk;       // filter extent of the dgrad operand: n_pad rounded up to 64
    int kr;       // column rows of the dgrad product: k_pad rounded up to 128
    int mc;       // pixels per chunk (multiple of 256)
    uint32_t plane_mul, plane_sh, ohw_mul, ohw_sh, ow_mul, ow_sh;  // multiply-shift divisors
    long long x_chw, thw;  // elements per input image, per input channel
    int hw;
    int split_mask;        // tap-mask encoding of the gather table (see tap_mask)
    const uint2* table;    // the plan's gather table: [k_pad] {x offset from the window origin, tap bits}
    size_t slab_wg_bytes;  // workspace of the slab weight gradient (0: gathered weight gradient)
    int* status;           // device status word (the debug build's index checks)
};

inline void divisor(uint32_t d, uint32_t& mul, uint32_t& sh)
{
    sh = 0;
    while ((1ull << sh) < d) ++sh;
    mul = (uint32_t)((((1ull << sh) - d) << 32) / d + 1);
}

// Output pixel m -> (n, ot, oh, ow), by multiply-shift division (m < 2^31).
SADMM_DEV uint32_t udiv(uint32_t n, uint32_t mul, uint32_t sh) { return (__umulhi(n, mul) + n) >> sh; }

SADMM_DEV void pixel_of(const BwdGeo& b, long long m, int& n, int& ot, int& oh, int& ow)
{
    const uint32_t mu = (uint32_t)m;
    n = (int)udiv(mu, b.plane_mul, b.plane_sh);
    const uint32_t p = mu - (uint32_t)n * (uint32_t)b.plane;
    ot = (int)udiv(p, b.ohw_mul, b.ohw_sh);
    const uint32_t r = p - (uint32_t)ot * (uint32_t)(b.OH * b.OW);
    oh = (int)udiv(r, b.ow_mul, b.ow_sh);
    ow = (int)(r - (uint32_t)oh * (uint32_t)b.OW);
}

// Packed columns per block of k_bwd_im2col / k_bwd_col2im: their gather-table
// entries sit in shared memory, and each thread decodes its pixel once for all.
constexpr int kTableCols = 32;

// A_T[j][ml] = x at packed column j of output pixel m0 + ml, through the plan's
// gather table (the column's x offset from the pixel's window origin, its tap
// bits tested against the pixel's tap mask); 0 outside the input, for padding
// columns and past the last pixel.  Block (bx, by): columns by*32 .. by*32+31.
__global__ void __launch_bounds__(256) k_bwd_im2col(const BwdGeo b, int g, long long m0, __nv_bfloat16* at)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ uint2 s_t[kTableCols];
    const int j0 = blockIdx.y * kTableCols;
    if (threadIdx.x < kTableCols) {
        const int j = j0 + threadIdx.x;
        s_t[threadIdx.x] = j < b.k_pad ? __ldg(b.table + j) : make_uint2(0u, 1u << 31);
    }
    __syncthreads();
    const int nj = min(kTableCols, b.k_pad - j0);
    const unsigned short* xs = reinterpret_cast<const unsigned short*>(b.x);
    unsigned short* as = reinterpret_cast<unsigned short*>(at);
    for (int ml = blockIdx.x * 256 + threadIdx.x; ml < b.mc; ml += gridDim.x * 256) {
        const long long m = m0 + ml;
        uint32_t M = 0;  // no tap is valid past the last pixel (tap bits are never 0)
        long long base = 0;
        if (m < b.M) {
            int n, ot, oh, ow;
            pixel_of(b, m, n, ot, oh, ow);
            const int it0 = ot * b.st - b.pt, ih0 = oh * b.sh - b.ph, iw0 = ow * b.sw - b.pw;
            M = tap_mask(it0, ih0, iw0, b.KT, b.KH, b.KW, b.T, b.H, b.W, b.split_mask);
            base = (long long)n * b.x_chw + (long long)g * b.Cg * b.thw + (long long)it0 * b.hw +
                   (long long)ih0 * b.W + iw0;
        }
        for (int jj = 0; jj < nj; ++jj) {
            const uint2 t = s_t[jj];
            as[(size_t)(j0 + jj) * b.mc + ml] =
                ((M & t.y) == t.y && dbg_in(base + (int)t.x, (long long)b.N * b.x_chw, b.status))
                    ? __ldg(xs + base + (int)t.x)
                    : (unsigned short)0;
        }
    }
}

SADMM_DEV float relu_grad(const BwdGeo& b, size_t off)
{
    if (!b.relu) return 1.0f;
    const float yv = (b.ydt == SADMM_BF16) ? __bfloat162float(static_cast<const __nv_bfloat16*>(b.y)[off])
                                           : static_cast<const float*>(b.y)[off];
    return yv > 0.0f ? 1.0f : 0.0f;
}

// dZ for the kept filters of group g and pixels m0 .. m0+mc-1, in two layouts:
// gt[i][ml] (filter-major, rows up to fr; for the weight gradient) and
// gm[ml][i] (pixel-major, i < fk; for the input gradient).  A null pointer
// skips that layout.
// Block (bx, by): pixels bx*64 .. +63 of the chunk, packed rows by*32 .. +31;
// the pixel-major copy goes out through a shared-memory transpose, 8 rows of a
// pixel per 16-byte store.
constexpr int kDyPix = 64, kDyRows = 32;

__global__ void __launch_bounds__(256) k_bwd_gather_dy(const BwdGeo b, int g, long long m0, __nv_bfloat16* gt,
                                                       __nv_bfloat16* gm)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ __nv_bfloat16 tile[kDyRows][kDyPix + 2];
    const int i0 = blockIdx.y * kDyRows, p0 = blockIdx.x * kDyPix;
    const int pl = threadIdx.x & (kDyPix - 1), r0 = threadIdx.x / kDyPix;  // 64 pixels x 4 rows
    const int ml = p0 + pl;
    const long long m = m0 + ml;
    const bool valid = ml < b.mc && m < b.M;
    size_t pbase = 0;  // offset of the pixel in plane 0 of its image
    if (valid) {
        const uint32_t n = udiv((uint32_t)m, b.plane_mul, b.plane_sh);
        pbase = (size_t)n * b.F * b.plane + ((uint32_t)m - n * (uint32_t)b.plane);
    }
    for (int k = 0; k < kDyRows / 4; ++k) {
        const int r = r0 + 4 * k, i = i0 + r;
        float v = 0.0f;
        if (valid && i < b.n_pad) {
            const int f = __ldg(b.rowmap + (long long)g * b.n_pad + i);
            if (f >= 0) {
                const size_t off = pbase + (size_t)f * b.plane;
                v = __bfloat162float(b.dy[off]) * relu_grad(b, off);
            }
        }
        const __nv_bfloat16 h = __float2bfloat16_rn(v);
        tile[r][pl] = h;
        if (gt && i < b.fr && ml < b.mc) gt[(size_t)i * b.mc + ml] = h;
    }
    __syncthreads();
    const int pl2 = threadIdx.x >> 2, rq = (threadIdx.x & 3) * 8;  // pixel, first of its 8 rows
    const int ml2 = p0 + pl2;
    if (gm && ml2 < b.mc && i0 + rq < b.fk) {  // fk is a multiple of 64: all 8 rows are inside
        uint32_t w[4];
        for (int e = 0; e < 4; ++e)
            w[e] = (uint32_t)__bfloat16_as_ushort(tile[rq + 2 * e][pl2]) |
                   ((uint32_t)__bfloat16_as_ushort(tile[rq + 2 * e + 1][pl2]) << 16);
        *reinterpret_cast<uint4*>(gm + (size_t)ml2 * b.fk + i0 + rq) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// wpt[j][i] = Wp[g][i][j] (zero past n_pad / k_pad).
__global__ void __launch_bounds__(256) k_bwd_transpose_wp(const BwdGeo b, int g, const __nv_bfloat16* wp,
                                                          __nv_bfloat16* wpt)
{
    pdl_wait();  // after the kernel before it in the stream
    const int j = blockIdx.y;
    for (int i = blockIdx.x * 256 + threadIdx.x; i < b.fk; i += gridDim.x * 256) {
        __nv_bfloat16 v = __float2bfloat16_rn(0.0f);
        if (j < b.k_pad && i < b.n_pad) v = wp[((size_t)g * b.n_pad + i) * b.k_pad + j];
        wpt[(size_t)j * b.fk + i] = v;
    }
}

// dx += dA at every valid (packed column, output pixel) position, through the
// gather table as in k_bwd_im2col; fp32 atomics (several pixels' windows
// overlap), zeros skipped.
__global__ void __launch_bounds__(256) k_bwd_col2im(const BwdGeo b, int g, long long m0, const float* dat, float* dx)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ uint2 s_t[kTableCols];
    const int j0 = blockIdx.y * kTableCols;
    if (threadIdx.x < kTableCols) {
        const int j = j0 + threadIdx.x;
        s_t[threadIdx.x] = j < b.k_pad ? __ldg(b.table + j) : make_uint2(0u, 1u << 31);
    }
    __syncthreads();
    const int nj = min(kTableCols, b.k_pad - j0);
    for (int ml = blockIdx.x * 256 + threadIdx.x; ml < b.mc; ml += gridDim.x * 256) {
        const long long m = m0 + ml;
        if (m >= b.M) break;
        int n, ot, oh, ow;
        pixel_of(b, m, n, ot, oh, ow);
        const int it0 = ot * b.st - b.pt, ih0 = oh * b.sh - b.ph, iw0 = ow * b.sw - b.pw;
        const uint32_t M = tap_mask(it0, ih0, iw0, b.KT, b.KH, b.KW, b.T, b.H, b.W, b.split_mask);
        const long long base = (long long)n * b.x_chw + (long long)g * b.Cg * b.thw + (long long)it0 * b.hw +
                               (long long)ih0 * b.W + iw0;
        for (int jj = 0; jj < nj; ++jj) {
            const uint2 t = s_t[jj];
            if ((M & t.y) == t.y) {
                const float v = dat[(size_t)(j0 + jj) * b.mc + ml];
                if (v != 0.0f && dbg_in(base + (int)t.x, (long long)b.N * b.x_chw, b.status))
                    atomicAdd(dx + base + (int)t.x, v);
            }
        }
    }
}

// dW[f_i][col_j] = sum over the pixel splits z, in order, of dws[z][i][j] for
// the kept pairs of conv group g (dW zeroed before): deterministic.
__global__ void __launch_bounds__(256) k_bwd_reduce_dw(const BwdGeo b, int g, const float* dws, int nsplit, float* dW)
{
    pdl_wait();  // after the kernel before it in the stream
    const int i = blockIdx.y;
    const int f = __ldg(b.rowmap + (long long)g * b.n_pad + i);
    if (f < 0) return;
    const long long K = (long long)b.Cg * b.taps;
    const size_t slice = (size_t)b.fr * b.k_pad;
    for (int j = blockIdx.x * 256 + threadIdx.x; j < b.n_cols; j += gridDim.x * 256) {
        const int col = __ldg(b.colidx + j);
        if (col < 0) continue;
        float acc = 0.0f;
        for (int z = 0; z < nsplit; ++z) acc += dws[z * slice + (size_t)i * b.k_pad + j];
        dW[(long long)f * K + col] = acc;
    }
}

// Bias gradient in two fixed-order stages.  Block (f, sl): the sum of dZ over
// every pixel of images sl, sl + S, ... (S = gridDim.y), 0 for a pruned filter.
constexpr int kDbSlices = 64;

__global__ void __launch_bounds__(256) k_bwd_db_part(const BwdGeo b, float* part)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ float red[256];
    const int f = blockIdx.x;
    const int g = f / b.Fg;
    // kept?  rowmap of group g lists the kept filters
    bool kept = false;
    const int cnt = __ldg(b.counts + 2 * g);
    for (int i = threadIdx.x; i < cnt; i += 256)
        if (__ldg(b.rowmap + (long long)g * b.n_pad + i) == f) kept = true;
    kept = __syncthreads_or(kept);
    float s = 0.0f;
    if (kept) {
        for (int n = blockIdx.y; n < b.N; n += gridDim.y) {
            const size_t base = ((size_t)n * b.F + f) * b.plane;  // the plane is contiguous
            for (int p = threadIdx.x; p < b.plane; p += 256)
                s += __bfloat162float(b.dy[base + p]) * relu_grad(b, base + p);
        }
    }
    red[threadIdx.x] = s;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) part[(size_t)f * gridDim.y + blockIdx.y] = red[0];
}

// db[f] = sum over the S slices, in order, of the partial sums.
__global__ void __launch_bounds__(256) k_bwd_db_final(const float* part, int F, int S, float* db)
{
    pdl_wait();  // after the kernel before it in the stream
    const int f = blockIdx.x * 256 + threadIdx.x;
    if (f >= F) return;
    float acc = 0.0f;
    for (int sl = 0; sl < S; ++sl) acc += part[(size_t)f * S + sl];
    db[f] = acc;
}

__global__ void __launch_bounds__(256) k_bwd_zero(float* p, long long n)
{
    pdl_wait();  // after the kernel before it in the stream
    for (long long i = (long long)blockIdx.x * 256 + threadIdx.x; i < n; i += (long long)gridDim.x * 256) p[i] = 0.0f;
}

inline long long rup(long long x, long long a) { return (x + a - 1) / a * a; }

struct Layout {
    size_t at, gt, gm, wpt, dat, dws, dbp, wsl, total;
};

int pick_bn(long long n);

// The weight gradient has only fr/128 x k_pad/bn output tiles, so each chunk's
// pixels (the GEMM's K) are split over enough CTAs to fill the GPU: about
// kWgradCtas CTAs in all, the split count a divisor of the chunk's 64-pixel
// stages.  Fixed (not the device's SM count) so that the workspace size is.
constexpr long long kWgradCtas = 256;

int wgrad_splits(const BwdGeo& b)
{
    const long long wtiles = (long long)(b.fr / 128) * (b.k_pad / pick_bn(b.k_pad));
    const long long nk = b.mc / 64;
    const long long want = std::max<long long>(1, kWgradCtas / std::max<long long>(wtiles, 1));
    for (long long d = std::min(want, nk); d >= 1; --d)
        if (nk % d == 0) return (int)d;
    return 1;
}

Layout layout(const BwdGeo& b)
{
    Layout l;
    size_t off = 0;
    auto take = [&off](size_t bytes) {
        const size_t at = off;
        off += (size_t)rup((long long)bytes, 1024);
        return at;
    };
    l.at = take((size_t)b.k_pad * b.mc * 2);
    l.gt = take((size_t)b.fr * b.mc * 2);
    l.gm = take((size_t)b.mc * b.fk * 2);
    l.wpt = take((size_t)b.kr * b.fk * 2);
    l.dat = take((size_t)b.kr * b.mc * 4);
    l.dws = take((size_t)wgrad_splits(b) * b.fr * b.k_pad * 4);  // [split][fr][k_pad]
    l.dbp = take((size_t)b.F * kDbSlices * 4);                    // [F][slices] bias-gradient partials
    l.wsl = take(b.slab_wg_bytes);                                // slab weight gradient (bwd_slab.cu)
    l.total = off;
    return l;
}

// Output pixels per chunk: the whole layer up to kBwdMaxChunk (the default
// workspace), or what a smaller workspace holds (at least 256).  A chunk's
// gathered operands and fp32 products (about 50 MB at 32768 pixels on AlexNet
// CONV1) stay in L2 from the kernel that writes them to the one that reads
// them; whole-layer chunks measured slower on GB300 (CONV1 1.60 -> 1.84 ms,
// CONV2 0.86 -> 1.54 ms at batch 128).
constexpr long long kBwdMaxChunk = 32768;

BwdGeo geometry(const sadmm_plan* plan, const Geometry& g, long long chunk)
{
    BwdGeo b;
    memset(&b, 0, sizeof(b));
    b.N = (int)g.n; b.C = (int)g.c; b.T = (int)g.t; b.H = (int)g.h; b.W = (int)g.w; b.F = (int)g.f;
    b.Cg = (int)g.cg; b.Fg = (int)g.fg; b.groups = (int)g.groups;
    b.KT = (int)g.kt; b.KH = (int)g.kh; b.KW = (int)g.kw;
    b.st = (int)g.st; b.sh = (int)g.sh; b.sw = (int)g.sw; b.pt = (int)g.pt; b.ph = (int)g.ph; b.pw = (int)g.pw;
    b.OT = (int)g.ot; b.OH = (int)g.oh; b.OW = (int)g.ow; b.plane = (int)g.plane; b.taps = (int)g.taps;
    b.M = g.m;
    b.n_pad = plan->n_pad;
    b.k_pad = plan->k_pad;
    b.n_cols = plan->n_cols;
    b.fr = (int)rup(plan->n_pad, 128);
    b.fk = (int)rup(plan->n_pad, 64);
    b.kr = (int)rup(plan->k_pad, 128);
    b.mc = (int)std::min<long long>(rup(g.m, 256), std::max<long long>(256, std::min(rup(chunk, 256), kBwdMaxChunk)));
    divisor((uint32_t)b.plane, b.plane_mul, b.plane_sh);
    divisor((uint32_t)(b.OH * b.OW), b.ohw_mul, b.ohw_sh);
    divisor((uint32_t)b.OW, b.ow_mul, b.ow_sh);
    b.x_chw = g.c * g.t * g.h * g.w;
    b.status = device_status_ptr();
    b.thw = g.t * g.h * g.w;
    b.hw = (int)(g.h * g.w);
    b.split_mask = tap_mask_mode(g);
    b.slab_wg_bytes = wgrad_slab_bytes(plan, g);
    return b;
}

int pick_bn(long long n)
{
    for (int bn = 256; bn >= 16; bn -= 16)
        if (n % bn == 0) return bn;
    return 16;
}

}  // namespace

size_t bwd_workspace_bytes(const sadmm_plan* plan, const Geometry& g, long long chunk)
{
    return layout(geometry(plan, g, chunk > 0 ? chunk : kBwdMaxChunk)).total;
}

// The largest chunk (a multiple of 256 pixels, at most the layer or
// kBwdMaxChunk) whose workspace fits ws_bytes; 0 when not even 256 pixels fit.
long long bwd_chunk_for(const sadmm_plan* plan, const Geometry& g, size_t ws_bytes)
{
    // The layout is not monotonic in the chunk (the weight-gradient split
    // count, and so its partial-sum slices, follows the chunk's divisors), so
    // every candidate from the largest down is checked: at most 128 of them.
    for (long long c = std::min<long long>(rup(g.m, 256), kBwdMaxChunk) / 256; c >= 1; --c)
        if (layout(geometry(plan, g, c * 256)).total <= ws_bytes) return c * 256;
    return 0;
}

sadmm_status launch_conv_bwd(const sadmm_plan* plan, const Geometry& g, const void* x, const void* dy, const void* y,
                             int ydt, int relu, float* dW, float* db, float* dx, void* ws, size_t ws_bytes,
                             cudaStream_t s)
{
    if (g.m >= (1ll << 31)) return SADMM_EUNSUPPORTED;  // pixel indices decode in 32 bits
    const long long chunk = bwd_chunk_for(plan, g, ws_bytes);
    if (chunk <= 0) return SADMM_EINVAL;
    BwdGeo b = geometry(plan, g, chunk);
    if (layout(b).total > ws_bytes) return SADMM_EINVAL;
    const char* base = static_cast<const char*>(plan->dev);
    b.x = static_cast<const __nv_bfloat16*>(x);
    b.dy = static_cast<const __nv_bfloat16*>(dy);
    b.y = y;
    b.ydt = ydt;
    b.relu = relu ? 1 : 0;
    b.rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    b.colidx = reinterpret_cast<const int*>(base + plan->off_colidx);
    b.counts = reinterpret_cast<const int*>(base + plan->off_counts);
    b.table = reinterpret_cast<const uint2*>(base + plan->off_gather);
    const __nv_bfloat16* wp = reinterpret_cast<const __nv_bfloat16*>(base + plan->off_wp);
    const Layout l = layout(b);
    char* w = static_cast<char*>(ws);
    __nv_bfloat16* at = reinterpret_cast<__nv_bfloat16*>(w + l.at);
    __nv_bfloat16* gt = reinterpret_cast<__nv_bfloat16*>(w + l.gt);
    __nv_bfloat16* gm = reinterpret_cast<__nv_bfloat16*>(w + l.gm);
    __nv_bfloat16* wpt = reinterpret_cast<__nv_bfloat16*>(w + l.wpt);
    float* dat = reinterpret_cast<float*>(w + l.dat);
    float* dws = reinterpret_cast<float*>(w + l.dws);
    float* dbp = reinterpret_cast<float*>(w + l.dbp);
    // table-driven im2col / col2im: one pixel per thread, 32 packed columns per block
    const unsigned tblocks = (unsigned)((b.mc + 255) / 256);
    const unsigned tcols = (unsigned)((b.k_pad + kTableCols - 1) / kTableCols);
    const long long K = g.cg * g.taps;

    if (dW) launch_pdl(k_bwd_zero, dim3(1024), dim3(256), 0, s, dW, g.f * K);
    // an input-slab plan's weight gradient runs on its slab, not through im2col
    const bool slab_dw = dW && b.slab_wg_bytes > 0;
    float* gdW = slab_dw ? nullptr : dW;  // the gathered weight gradient's output
    if (slab_dw) {
        const sadmm_status sst = launch_wgrad_slab(plan, g, x, dy, y, ydt, relu, dW, w + l.wsl, s);
        if (sst != SADMM_OK) return sst;
    }
    const int wbn = pick_bn(b.k_pad);
    const int wsplit = wgrad_splits(b);
    if (dx) launch_pdl(k_bwd_zero, dim3(2048), dim3(256), 0, s, dx, g.n * g.c * g.t * g.h * g.w);
    if (db) {
        const int slices = (int)std::min<long long>(g.n, kDbSlices);
        launch_pdl(k_bwd_db_part, dim3((unsigned)g.f, (unsigned)slices), dim3(256), 0, s, b, dbp);
        launch_pdl(k_bwd_db_final, dim3((unsigned)((g.f + 255) / 256)), dim3(256), 0, s,
                   static_cast<const float*>(dbp), (int)g.f, slices, db);
    }
    sadmm_status st = SADMM_OK;
    for (int grp = 0; grp < b.groups && st == SADMM_OK; ++grp) {
        if (dx)
            launch_pdl(k_bwd_transpose_wp, dim3((unsigned)((b.fk + 255) / 256), (unsigned)b.kr), dim3(256), 0, s, b,
                       grp, wp, wpt);
        for (long long m0 = 0; (gdW || dx) && m0 < g.m && st == SADMM_OK; m0 += b.mc) {
            const unsigned dyrows = (unsigned)std::max(gdW ? b.fr : 0, dx ? b.fk : 0);
            launch_pdl(k_bwd_gather_dy, dim3((unsigned)((b.mc + kDyPix - 1) / kDyPix), (dyrows + kDyRows - 1) / kDyRows),
                       dim3(256), 0, s, b, grp, m0, gdW ? gt : nullptr, dx ? gm : nullptr);
            if (gdW) {
                launch_pdl(k_bwd_im2col, dim3(tblocks, tcols), dim3(256), 0, s, b, grp, m0, at);
                // split z: dws[z][i][j] (+)= sum over its pixels m of gt[i][m] * at[j][m]
                st = launch_gemm(gt, at, dws, b.fr, b.k_pad, b.mc, b.k_pad, wbn, m0 > 0, s, wsplit,
                                 (long long)b.fr * b.k_pad);
            }
            if (dx && st == SADMM_OK) {
                // dat[j][m] = sum_i wpt[j][i] * gm[m][i]
                st = launch_gemm(wpt, gm, dat, b.kr, b.mc, b.fk, b.mc, pick_bn(b.mc), false, s);
                if (st == SADMM_OK)
                    launch_pdl(k_bwd_col2im, dim3(tblocks, tcols), dim3(256), 0, s, b, grp, m0,
                               static_cast<const float*>(dat), dx);
            }
        }
        if (gdW && st == SADMM_OK)
            launch_pdl(k_bwd_reduce_dw, dim3((unsigned)((b.k_pad + 255) / 256), (unsigned)b.n_pad), dim3(256), 0, s, b,
                       grp, static_cast<const float*>(dws), wsplit, dW);
    }
    if (st != SADMM_OK) return st;
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
