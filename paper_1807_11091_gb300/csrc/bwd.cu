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

// A_T[j][ml] = x at kept column j of output pixel m0 + ml (0 outside the input,
// for padding columns and past the last pixel).
__global__ void __launch_bounds__(256) k_bwd_im2col(const BwdGeo b, int g, long long m0, __nv_bfloat16* at)
{
    const int j = blockIdx.y;
    const int col = j < b.n_cols ? __ldg(b.colidx + j) : -1;
    int c = 0, kt = 0, kh = 0, kw = 0;
    if (col >= 0) {
        c = col / b.taps;
        const int r = col - c * b.taps;
        kt = r / (b.KH * b.KW);
        kh = (r / b.KW) % b.KH;
        kw = r % b.KW;
    }
    for (int ml = blockIdx.x * 256 + threadIdx.x; ml < b.mc; ml += gridDim.x * 256) {
        const long long m = m0 + ml;
        float v = 0.0f;
        if (col >= 0 && m < b.M) {
            int n, ot, oh, ow;
            pixel_of(b, m, n, ot, oh, ow);
            const int it = ot * b.st - b.pt + kt, ih = oh * b.sh - b.ph + kh, iw = ow * b.sw - b.pw + kw;
            if ((unsigned)it < (unsigned)b.T && (unsigned)ih < (unsigned)b.H && (unsigned)iw < (unsigned)b.W)
                v = __bfloat162float(b.x[((((long long)n * b.C + (long long)g * b.Cg + c) * b.T + it) * b.H + ih) *
                                             b.W + iw]);
        }
        at[(size_t)j * b.mc + ml] = __float2bfloat16_rn(v);
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
// gt[i][ml] (filter-major, rows up to fr) and gm[ml][i] (pixel-major, i < fk).
__global__ void __launch_bounds__(256) k_bwd_gather_dy(const BwdGeo b, int g, long long m0, __nv_bfloat16* gt,
                                                       __nv_bfloat16* gm)
{
    const int i = blockIdx.y;  // 0 .. max(fr, fk)-1
    const int f = i < b.n_pad ? __ldg(b.rowmap + (long long)g * b.n_pad + i) : -1;
    for (int ml = blockIdx.x * 256 + threadIdx.x; ml < b.mc; ml += gridDim.x * 256) {
        const long long m = m0 + ml;
        float v = 0.0f;
        if (f >= 0 && m < b.M) {
            const int n = (int)(m / b.plane);
            const size_t off = ((size_t)n * b.F + f) * b.plane + (size_t)(m - (long long)n * b.plane);
            v = __bfloat162float(b.dy[off]) * relu_grad(b, off);
        }
        const __nv_bfloat16 h = __float2bfloat16_rn(v);
        if (i < b.fr) gt[(size_t)i * b.mc + ml] = h;
        if (i < b.fk) gm[(size_t)ml * b.fk + i] = h;
    }
}

// wpt[j][i] = Wp[g][i][j] (zero past n_pad / k_pad).
__global__ void __launch_bounds__(256) k_bwd_transpose_wp(const BwdGeo b, int g, const __nv_bfloat16* wp,
                                                          __nv_bfloat16* wpt)
{
    const int j = blockIdx.y;
    for (int i = blockIdx.x * 256 + threadIdx.x; i < b.fk; i += gridDim.x * 256) {
        __nv_bfloat16 v = __float2bfloat16_rn(0.0f);
        if (j < b.k_pad && i < b.n_pad) v = wp[((size_t)g * b.n_pad + i) * b.k_pad + j];
        wpt[(size_t)j * b.fk + i] = v;
    }
}

// dx += col2im(dA): dat[j][ml] for kept column j of pixel m0 + ml.
__global__ void __launch_bounds__(256) k_bwd_col2im(const BwdGeo b, int g, long long m0, const float* dat, float* dx)
{
    const int j = blockIdx.y;
    const int col = j < b.n_cols ? __ldg(b.colidx + j) : -1;
    if (col < 0) return;
    const int c = col / b.taps;
    const int r = col - c * b.taps;
    const int kt = r / (b.KH * b.KW), kh = (r / b.KW) % b.KH, kw = r % b.KW;
    for (int ml = blockIdx.x * 256 + threadIdx.x; ml < b.mc; ml += gridDim.x * 256) {
        const long long m = m0 + ml;
        if (m >= b.M) break;
        int n, ot, oh, ow;
        pixel_of(b, m, n, ot, oh, ow);
        const int it = ot * b.st - b.pt + kt, ih = oh * b.sh - b.ph + kh, iw = ow * b.sw - b.pw + kw;
        if ((unsigned)it < (unsigned)b.T && (unsigned)ih < (unsigned)b.H && (unsigned)iw < (unsigned)b.W) {
            const float v = dat[(size_t)j * b.mc + ml];
            if (v != 0.0f)
                atomicAdd(dx + ((((long long)n * b.C + (long long)g * b.Cg + c) * b.T + it) * b.H + ih) * b.W + iw,
                          v);
        }
    }
}

// dW[f_i][col_j] = dWp[g][i][j] for kept pairs (dW zeroed before).
__global__ void __launch_bounds__(256) k_bwd_scatter_dw(const BwdGeo b, int g, const float* dwp, float* dW)
{
    const int i = blockIdx.y;
    const int f = __ldg(b.rowmap + (long long)g * b.n_pad + i);
    if (f < 0) return;
    const long long K = (long long)b.Cg * b.taps;
    for (int j = blockIdx.x * 256 + threadIdx.x; j < b.n_cols; j += gridDim.x * 256) {
        const int col = __ldg(b.colidx + j);
        if (col >= 0) dW[(long long)f * K + col] = dwp[(size_t)i * b.k_pad + j];
    }
}

// db[f] = sum over images and pixels of dZ (fixed order), 0 for pruned filters.
__global__ void __launch_bounds__(256) k_bwd_db(const BwdGeo b, float* db)
{
    __shared__ float part[256];
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
        for (long long m = threadIdx.x; m < b.M; m += 256) {
            const int n = (int)(m / b.plane);
            const size_t off = ((size_t)n * b.F + f) * b.plane + (size_t)(m - (long long)n * b.plane);
            s += __bfloat162float(b.dy[off]) * relu_grad(b, off);
        }
    }
    part[threadIdx.x] = s;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) part[threadIdx.x] += part[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) db[f] = part[0];
}

__global__ void __launch_bounds__(256) k_bwd_zero(float* p, long long n)
{
    for (long long i = (long long)blockIdx.x * 256 + threadIdx.x; i < n; i += (long long)gridDim.x * 256) p[i] = 0.0f;
}

inline long long rup(long long x, long long a) { return (x + a - 1) / a * a; }

struct Layout {
    size_t at, gt, gm, wpt, dat, dwp, total;
};

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
    l.dwp = take((size_t)b.groups * b.fr * b.k_pad * 4);
    l.total = off;
    return l;
}

BwdGeo geometry(const sadmm_plan* plan, const Geometry& g)
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
    b.mc = (int)std::min<long long>(rup(g.m, 256), 32768);
    divisor((uint32_t)b.plane, b.plane_mul, b.plane_sh);
    divisor((uint32_t)(b.OH * b.OW), b.ohw_mul, b.ohw_sh);
    divisor((uint32_t)b.OW, b.ow_mul, b.ow_sh);
    return b;
}

int pick_bn(long long n)
{
    for (int bn = 256; bn >= 16; bn -= 16)
        if (n % bn == 0) return bn;
    return 16;
}

}  // namespace

size_t bwd_workspace_bytes(const sadmm_plan* plan, const Geometry& g)
{
    return layout(geometry(plan, g)).total;
}

sadmm_status launch_conv_bwd(const sadmm_plan* plan, const Geometry& g, const void* x, const void* dy, const void* y,
                             int ydt, int relu, float* dW, float* db, float* dx, void* ws, cudaStream_t s)
{
    if (g.m >= (1ll << 31)) return SADMM_EUNSUPPORTED;  // pixel indices decode in 32 bits
    BwdGeo b = geometry(plan, g);
    const char* base = static_cast<const char*>(plan->dev);
    b.x = static_cast<const __nv_bfloat16*>(x);
    b.dy = static_cast<const __nv_bfloat16*>(dy);
    b.y = y;
    b.ydt = ydt;
    b.relu = relu ? 1 : 0;
    b.rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    b.colidx = reinterpret_cast<const int*>(base + plan->off_colidx);
    b.counts = reinterpret_cast<const int*>(base + plan->off_counts);
    const __nv_bfloat16* wp = reinterpret_cast<const __nv_bfloat16*>(base + plan->off_wp);
    const Layout l = layout(b);
    char* w = static_cast<char*>(ws);
    __nv_bfloat16* at = reinterpret_cast<__nv_bfloat16*>(w + l.at);
    __nv_bfloat16* gt = reinterpret_cast<__nv_bfloat16*>(w + l.gt);
    __nv_bfloat16* gm = reinterpret_cast<__nv_bfloat16*>(w + l.gm);
    __nv_bfloat16* wpt = reinterpret_cast<__nv_bfloat16*>(w + l.wpt);
    float* dat = reinterpret_cast<float*>(w + l.dat);
    float* dwp = reinterpret_cast<float*>(w + l.dwp);
    const unsigned xblocks = (unsigned)std::min<long long>((b.mc + 255) / 256, 64);
    const long long K = g.cg * g.taps;

    if (dW) {
        k_bwd_zero<<<1024, 256, 0, s>>>(dW, g.f * K);
        k_bwd_zero<<<256, 256, 0, s>>>(dwp, (long long)b.groups * b.fr * b.k_pad);
    }
    // weight-gradient tiles are few (fr/128 x k_pad/bn): split the pixel
    // dimension of each chunk over enough CTAs to fill the GPU
    const int wbn = pick_bn(b.k_pad);
    const long long wtiles = (long long)(b.fr / 128) * (b.k_pad / wbn);
    int wsplit = 1;
    {
        const long long nk = b.mc / 64;
        long long want = std::max<long long>(1, (2LL * device_sm_count()) / std::max<long long>(wtiles, 1));
        for (long long d = std::min(want, nk); d >= 1; --d)
            if (nk % d == 0) { wsplit = (int)d; break; }
    }
    if (dx) k_bwd_zero<<<2048, 256, 0, s>>>(dx, g.n * g.c * g.t * g.h * g.w);
    if (db) k_bwd_db<<<(unsigned)g.f, 256, 0, s>>>(b, db);
    sadmm_status st = SADMM_OK;
    for (int grp = 0; grp < b.groups && st == SADMM_OK; ++grp) {
        float* dwp_g = dwp + (size_t)grp * b.fr * b.k_pad;
        if (dx) k_bwd_transpose_wp<<<dim3((unsigned)((b.fk + 255) / 256), (unsigned)b.kr), 256, 0, s>>>(b, grp, wp, wpt);
        for (long long m0 = 0; m0 < g.m && st == SADMM_OK; m0 += b.mc) {
            const unsigned dyrows = (unsigned)std::max(b.fr, b.fk);
            k_bwd_gather_dy<<<dim3(xblocks, dyrows), 256, 0, s>>>(b, grp, m0, gt, gm);
            if (dW) {
                k_bwd_im2col<<<dim3(xblocks, (unsigned)b.k_pad), 256, 0, s>>>(b, grp, m0, at);
                // dWp[i][j] += sum_m gt[i][m] * at[j][m] (zeroed above; split over pixels)
                st = launch_gemm(gt, at, dwp_g, b.fr, b.k_pad, b.mc, b.k_pad, wbn, true, s, wsplit);
            }
            if (dx && st == SADMM_OK) {
                // dat[j][m] = sum_i wpt[j][i] * gm[m][i]
                st = launch_gemm(wpt, gm, dat, b.kr, b.mc, b.fk, b.mc, pick_bn(b.mc), false, s);
                if (st == SADMM_OK)
                    k_bwd_col2im<<<dim3(xblocks, (unsigned)b.k_pad), 256, 0, s>>>(b, grp, m0, dat, dx);
            }
        }
        if (dW && st == SADMM_OK)
            k_bwd_scatter_dw<<<dim3((unsigned)((b.k_pad + 255) / 256), (unsigned)b.n_pad), 256, 0, s>>>(b, grp, dwp_g,
                                                                                                     dW);
    }
    if (st != SADMM_OK) return st;
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
