// conv_common.cuh -- pieces shared by the two forward kernels (conv_fwd.cu,
// the gathered implicit GEMM, and conv_slab.cu, the input-slab path): the
// invariant-divisor division and the epilogue's bias / ReLU / store step.
#pragma once

#include "common.cuh"

namespace sadmm {
namespace {

constexpr int kEpiCols = 16;  // accumulator columns per epilogue TMEM load

// Division of a non-negative int below 2^31 by an invariant divisor d >= 1:
// q = (umulhi(n, mul) + n) >> shift with shift = ceil(log2 d) and
// mul = floor(2^32 (2^shift - d) / d) + 1 (the round-up method of Granlund
// and Montgomery); umulhi(n, mul) <= n, so the sum stays below 2^32.
struct FastDiv {
    uint32_t d, mul, shift;
};

inline FastDiv make_fastdiv(uint32_t d)
{
    FastDiv f;
    f.d = d;
    uint32_t s = 0;
    while ((1ull << s) < d) ++s;
    f.shift = s;
    f.mul = (uint32_t)((((1ull << s) - d) << 32) / d + 1);
    return f;
}

SADMM_DEV uint32_t fdiv(uint32_t n, const FastDiv& f) { return (__umulhi(n, f.mul) + n) >> f.shift; }

// The output's extent for the debug build's store checks: yf / yh point at
// element pix of y, which holds total elements.
struct YCheck {
    long long pix, total;
    int* status;
};
SADMM_DEV bool y_ok(const YCheck& c, long long off) { return dbg_in(c.pix + off, c.total, c.status); }

// Bias, ReLU and the stores of accumulator columns c0 .. c0+kEpiCols-1 of one
// pixel (columns at or past nrows are skipped): t_off / t_bias give each
// column's output-plane offset and bias, yf / yh point at the pixel in plane 0.
template <bool OUT_BF16>
SADMM_DEV void store_cols(const float (&v)[kEpiCols], int c0, int nrows, const int* t_off, const float* t_bias,
                          int relu, float* yf, __nv_bfloat16* yh, const YCheck& yc)
{
    if (c0 + kEpiCols <= nrows) {
#pragma unroll
        for (int j = 0; j < kEpiCols; j += 4) {
            const int4 o = *reinterpret_cast<const int4*>(t_off + c0 + j);
            const float4 b = *reinterpret_cast<const float4*>(t_bias + c0 + j);
            float v0 = v[j] + b.x, v1 = v[j + 1] + b.y, v2 = v[j + 2] + b.z, v3 = v[j + 3] + b.w;
            if (relu) {
                v0 = fmaxf(v0, 0.0f); v1 = fmaxf(v1, 0.0f);
                v2 = fmaxf(v2, 0.0f); v3 = fmaxf(v3, 0.0f);
            }
            if (OUT_BF16) {
                if (y_ok(yc, o.x)) yh[o.x] = __float2bfloat16_rn(v0);
                if (y_ok(yc, o.y)) yh[o.y] = __float2bfloat16_rn(v1);
                if (y_ok(yc, o.z)) yh[o.z] = __float2bfloat16_rn(v2);
                if (y_ok(yc, o.w)) yh[o.w] = __float2bfloat16_rn(v3);
            } else {
                if (y_ok(yc, o.x)) __stcs(yf + o.x, v0);
                if (y_ok(yc, o.y)) __stcs(yf + o.y, v1);
                if (y_ok(yc, o.z)) __stcs(yf + o.z, v2);
                if (y_ok(yc, o.w)) __stcs(yf + o.w, v3);
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < kEpiCols; ++j) {
            if (c0 + j < nrows) {
                float x = v[j] + t_bias[c0 + j];
                if (relu) x = fmaxf(x, 0.0f);
                const int off = t_off[c0 + j];
                if (!y_ok(yc, off)) continue;
                if (OUT_BF16)
                    yh[off] = __float2bfloat16_rn(x);
                else
                    __stcs(yf + off, x);
            }
        }
    }
}

}  // namespace
}  // namespace sadmm
