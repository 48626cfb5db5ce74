// project.cu -- Euclidean projection onto a structured-sparsity set (Sec. 4,
// solution of the Z-subproblem, Eq. 4): squared Frobenius norms of the filter,
// channel or shape groups of V = W (+U), then an exact top-k.
//
// Every launch serves a batch of layers (a single call is a batch of one):
// the layers' parameters travel in kernel parameter space, and a block finds
// its layer by its index.
//   k_filter_keys   one block per GEMM row (filter), or a warp per row for
//                   rows of at most 1024 columns: error-free fp32 pair sums of
//                   squares (SqSum) over 16-byte loads, warp-shuffle and
//                   fixed-order block reduction.
//   k_column_keys   32 columns per block, 8 warps over the (kept) rows, fixed
//                   order shared-memory reduction: one key per GEMM column.
//   k_select_rows / k_select_cols
//                   one block per layer: optional channel sums of column keys,
//                   an MSB-first radix select over the fp64 key bit patterns
//                   (exact k-th largest key), then an ordered compaction that
//                   keeps every key above it and the lowest-index keys equal
//                   to it.  The layers' selects run side by side.
//
// Keys are non-negative fp64 values, so their IEEE bit patterns order like the
// values; selection compares bit patterns (a NaN key would rank above +Inf).
#include <string.h>

#include <algorithm>
#include <atomic>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

template <typename T>
SADMM_DEV float to_f32(T v);
template <>
SADMM_DEV float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }
template <>
SADMM_DEV float to_f32<float>(float v) { return v; }

// A sum of squares V_e^2 kept on the fp32 pipe (fp64 arithmetic is slow on
// this GPU) without losing precision: V = W (+U) is formed as an exact pair
// s + err (TwoSum), its square as p + e with p = s*s and
// e = fma(s, s, -p) + 2*s*err (exact up to err^2 <= 2^-48 V^2); the running
// sum hi collects p, each addition's exact rounding error (TwoSum) goes to lo
// with e, and every 8 terms the pair is renormalised (hi + lo exactly, lo below
// half an ulp of hi).  The lo additions between renormalisations bound the
// relative error of a thread's sum by about 8^2 * 2^-48 = 2^-42; pair merges
// across threads add about 2^-47 each.  Elements with |s| outside
// [2^-40, 2^40] (whose squares or residuals could leave fp32's normal range)
// are squared and added in fp64 (d) instead.
SADMM_DEV void two_sum(float a, float b, float& s, float& e)
{
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

struct SqSum {
    float hi, lo;
    double d;
    int n;
    SADMM_DEV void init()
    {
        hi = lo = 0.0f;
        d = 0.0;
        n = 0;
    }
    SADMM_DEV void renorm()
    {
        const float t = hi + lo;
        lo = lo - (t - hi);
        hi = t;
    }
    template <typename T>
    SADMM_DEV void add(const T* __restrict__ W, const T* __restrict__ U, long long i)
    {
        add_f(to_f32<T>(W[i]), U ? to_f32<T>(U[i]) : 0.0f, U != nullptr);
    }
    // adds V^2 for V = w (+ u when has_u)
    SADMM_DEV void add_f(float w, float u, bool has_u)
    {
        float sv = w, err = 0.0f;
        if (has_u) two_sum(w, u, sv, err);
        const float as = fabsf(sv);
        if (as >= 0x1p-40f && as <= 0x1p40f) {
            const float p = sv * sv;
            const float e = fmaf(sv, sv, -p) + 2.0f * sv * err;
            float t, te;
            two_sum(hi, p, t, te);
            lo += te + e;
            hi = t;
            if (++n == 8) {
                renorm();
                n = 0;
            }
        } else if (sv != 0.0f || err != 0.0f) {
            const double v = (double)w + (double)u;
            d = fma(v, v, d);
        }
    }
    // adds another sum given as its pair (and fp64 part)
    SADMM_DEV void merge(float ohi, float olo, double od)
    {
        float t, te;
        two_sum(hi, ohi, t, te);
        lo += olo + te;
        hi = t;
        renorm();
        d += od;
    }
    // the warp's sums merged into lane 0 in a fixed order (lane 0's result
    // is the warp total; d is reduced only when some lane has an fp64 part)
    SADMM_DEV void warp_reduce()
    {
        renorm();
        const bool any_d = __any_sync(0xffffffffu, d != 0.0);
        for (int o = 16; o > 0; o >>= 1) {
            const float oh = __shfl_down_sync(0xffffffffu, hi, o);
            const float ol = __shfl_down_sync(0xffffffffu, lo, o);
            const double od = any_d ? __shfl_down_sync(0xffffffffu, d, o) : 0.0;
            merge(oh, ol, od);
        }
    }
    SADMM_DEV double value() const { return ((double)hi + (double)lo) + d; }
};

// Eight consecutive elements as fp32, from a 16-byte aligned address.
SADMM_DEV void load8(const __nv_bfloat16* p, float (&v)[8])
{
    const uint4 q = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        v[2 * i] = __uint_as_float(w[i] << 16);
        v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}
SADMM_DEV void load8(const float* p, float (&v)[8])
{
    const float4 a = __ldg(reinterpret_cast<const float4*>(p));
    const float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Adds the squares of a row's K elements: thread t of nt takes the 8-element
// runs t, t + nt, ... with 16-byte loads when the row (of W, and of U) starts
// 16-byte aligned, then the last K % 8 elements one by one (K8 + t, ...);
// every element one by one when the row is not aligned.
template <typename T>
SADMM_DEV void add_row(SqSum& acc, const T* __restrict__ Wr, const T* __restrict__ Ur, int K, int t, int nt)
{
    const bool vec = ((reinterpret_cast<uintptr_t>(Wr) | reinterpret_cast<uintptr_t>(Ur)) & 15) == 0;
    const int K8 = vec ? (K & ~7) : 0;
    for (int k = t * 8; k < K8; k += nt * 8) {
        float w[8], u[8];
        load8(Wr + k, w);
        if (Ur) load8(Ur + k, u);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc.add_f(w[e], Ur ? u[e] : 0.0f, Ur != nullptr);
    }
    for (int k = K8 + t; k < K; k += nt) acc.add(Wr, Ur, k);
}

// Per-layer parameters of a batched projection (kernel parameter space; a
// block finds its layer by its first-block offsets).
struct BLayer {
    const void* W;
    const void* U;
    const int* krows;  // kept-row list the column keys sum over (NULL: every row)
    int* filt_idx;
    int* col_idx;
    double* keys_out;
    double* fkeys;  // filter keys [F]
    double* ckeys;  // column-group keys [G]
    double* parts;  // partial column keys [R][K]
    uint8_t* rkeep;
    uint8_t* ckeep;
    int F, K, taps, G, k_filters, k_cols;
    int do_rows, do_cols;  // 1: keys and select of this kind run
    int R, cblocks, nrows;
    int fk0, ck0, ka0, ka_n;  // first block in the filter-key, column-key, keep-all grids; keep-all length
    int rpb;                  // filter-key rows per block: 8 (a warp per row, K <= 1024) or 1
    int rows_all, cols_all;   // lists written whole by the keep-all pass
};

struct BatchArgs {
    int n;
    int fk_total;  // blocks of the filter-key pass; the keep-all blocks follow them
    BLayer L[kMaxBatch];
};

// The layer whose block range of one grid holds block b: the last layer with
// first block <= b (the ranges are ascending; empty ranges are skipped by the
// callers' bounds checks).
template <int BLayer::*Start>
SADMM_DEV int find_layer(const BatchArgs& a, int b)
{
    int lo = 0, hi = a.n - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (a.L[mid].*Start <= b) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// Index lists 0..n-1 and keep flags of one for the kinds kept whole: block b
// of the keep-all range.
SADMM_DEV void keep_all_block(const BatchArgs& ba, int b)
{
    const int l = find_layer<&BLayer::ka0>(ba, b);
    const BLayer& L = ba.L[l];
    const int i = (b - L.ka0) * 256 + threadIdx.x;
    if (i >= L.ka_n) return;
    if (L.rows_all && i < L.F) {
        L.filt_idx[i] = i;
        if (L.rkeep) L.rkeep[i] = 1;
    }
    if (L.cols_all && i < L.G) {
        L.col_idx[i] = i;
        if (L.ckeep) L.ckeep[i] = 1;
    }
}

// O_a = sum_k V[a,k]^2 for every row a (filter-wise groups): one block per
// row of every layer that needs them, a sum of squares per thread (SqSum),
// fixed-order warp and block merges.  Blocks past the filter-key range write
// the index lists of the kinds kept whole.
template <typename T>
__global__ void __launch_bounds__(256) k_filter_keys(const __grid_constant__ BatchArgs ba)
{
    pdl_wait();  // after the kernel before it in the stream
    if ((int)blockIdx.x >= ba.fk_total) {
        keep_all_block(ba, (int)blockIdx.x - ba.fk_total);
        return;
    }
    __shared__ float part_h[8], part_l[8];
    __shared__ double part_d[8];
    const int l = find_layer<&BLayer::fk0>(ba, blockIdx.x);
    const BLayer& L = ba.L[l];
    const T* W = static_cast<const T*>(L.W);
    const T* U = static_cast<const T*>(L.U);
    const int K = L.K;
    const int lane = threadIdx.x & 31, wy = threadIdx.x >> 5;
    if (L.rpb == 8) {
        // short rows: warp wy sums row 8 b + wy, lanes strided over its columns
        const int a = (blockIdx.x - L.fk0) * 8 + wy;
        if (!L.do_rows || a >= L.F) return;
        const long long base = (long long)a * K;
        SqSum acc;
        acc.init();
        add_row(acc, W + base, U ? U + base : nullptr, K, lane, 32);
        acc.warp_reduce();
        if (lane == 0) L.fkeys[a] = acc.value();
        return;
    }
    const int a = blockIdx.x - L.fk0;
    if (!L.do_rows || a >= L.F) return;
    const long long base = (long long)a * K;
    SqSum acc;
    acc.init();
    add_row(acc, W + base, U ? U + base : nullptr, K, (int)threadIdx.x, 256);
    acc.warp_reduce();
    if (lane == 0) {
        part_h[wy] = acc.hi;
        part_l[wy] = acc.lo;
        part_d[wy] = acc.d;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        SqSum t;
        t.init();
        for (int q = 0; q < 8; ++q) t.merge(part_h[q], part_l[q], part_d[q]);
        L.fkeys[a] = t.value();
    }
}

// Partial column keys: block (bx, by) of a layer sums V[a,j]^2 over rows by,
// by + R, ... of the kept-row list for the 32 columns j of bx, and writes
// part[by][j].  The select adds the R partials of a column in fixed order.
template <typename T>
__global__ void __launch_bounds__(256) k_column_keys(const __grid_constant__ BatchArgs ba)
{
    pdl_wait();  // after the kernel before it in the stream (the kept rows)
    __shared__ float part_h[8][33], part_l[8][33];
    __shared__ double part_d[8][33];
    const int l = find_layer<&BLayer::ck0>(ba, blockIdx.x);
    const BLayer& L = ba.L[l];
    const int local = blockIdx.x - L.ck0;
    if (!L.do_cols || local >= L.cblocks * L.R) return;
    const int bx = local % L.cblocks, by = local / L.cblocks;
    const T* W = static_cast<const T*>(L.W);
    const T* U = static_cast<const T*>(L.U);
    const int K = L.K, R = L.R;
    const int lane = threadIdx.x & 31;
    const int wy = threadIdx.x >> 5;
    const int j = bx * 32 + lane;
    SqSum acc;
    acc.init();
    if (j < K) {
        for (int r = by + R * wy; r < L.nrows; r += 8 * R) {
            const int a = L.krows ? L.krows[r] : r;
            acc.add(W, U, (long long)a * K + j);
        }
    }
    acc.renorm();
    part_h[wy][lane] = acc.hi;
    part_l[wy][lane] = acc.lo;
    part_d[wy][lane] = acc.d;
    __syncthreads();
    if (wy == 0 && j < K) {
        SqSum t;
        t.init();
        for (int q = 0; q < 8; ++q) t.merge(part_h[q][lane], part_l[q][lane], part_d[q][lane]);
        L.parts[(long long)by * K + j] = t.value();
    }
}

constexpr int kSelThreads = 1024;

// Exclusive block-wide prefix count of a predicate (1024 threads).  Returns
// the exclusive count for this thread; *total gets the block total.
SADMM_DEV int block_excl_count(bool pred, int* warp_tot, int* total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned b = __ballot_sync(0xffffffffu, pred);
    const int in_warp = __popc(b & ((1u << lane) - 1u));
    if (lane == 0) warp_tot[warp] = __popc(b);
    __syncthreads();
    if (warp == 0) {
        const int v = warp_tot[lane];
        int inc = v;
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += t;
        }
        warp_tot[lane] = inc - v;  // exclusive
        if (lane == 31) warp_tot[32] = inc;
    }
    __syncthreads();
    const int r = warp_tot[warp] + in_warp;
    *total = warp_tot[32];
    __syncthreads();  // warp_tot is reused by the next call
    return r;
}

// Exact top-k of G fp64 keys (ties to the lower index), ascending index list,
// by one block.  When taps > 1 the keys are first formed as sums of `taps`
// consecutive source keys (channel-wise groups from column keys), each the sum
// of its nparts partial sums.  keep_out (optional) gets a byte per group: 1
// when kept.
SADMM_DEV void select_block(const double* __restrict__ src, int G, int taps, int k, int nparts,
                            long long part_stride, double* __restrict__ keys, double* __restrict__ keys_out,
                            int* __restrict__ out_idx, uint8_t* __restrict__ keep_out)
{
    __shared__ unsigned int hist[256];
    __shared__ unsigned long long s_prefix;
    __shared__ int s_kk;
    __shared__ int s_done;
    __shared__ int warp_tot[33];
    const int tid = threadIdx.x;

    // 1. keys: the sum of the nparts partial sums of each source key, then of
    //    `taps` consecutive source keys (channel-wise groups); and the optional
    //    copy for the caller
    // the taps * nparts source values of key i, in four independent partial
    // sums (fixed order: entry e goes to partial e % 4)
    for (int i = tid; i < G; i += kSelThreads) {
        const int n = taps * nparts;
        double v0 = 0.0, v1 = 0.0, v2 = 0.0, v3 = 0.0;
        int e = 0;
        for (; e + 3 < n; e += 4) {
            const int t0 = e / nparts, t1 = (e + 1) / nparts, t2 = (e + 2) / nparts, t3 = (e + 3) / nparts;
            v0 += src[(e - t0 * nparts) * part_stride + (long long)i * taps + t0];
            v1 += src[(e + 1 - t1 * nparts) * part_stride + (long long)i * taps + t1];
            v2 += src[(e + 2 - t2 * nparts) * part_stride + (long long)i * taps + t2];
            v3 += src[(e + 3 - t3 * nparts) * part_stride + (long long)i * taps + t3];
        }
        for (; e < n; ++e) {
            const int t = e / nparts;
            v0 += src[(e - t * nparts) * part_stride + (long long)i * taps + t];
        }
        const double v = (v0 + v1) + (v2 + v3);
        if (taps > 1 || nparts > 1) keys[i] = v;
        if (keys_out) keys_out[i] = v;
    }
    const double* kv = (taps > 1 || nparts > 1) ? keys : src;
    __syncthreads();

    if (k <= 0 || k >= G) {
        for (int i = tid; i < G; i += kSelThreads) {
            if (k >= G) out_idx[i] = i;
            if (keep_out) keep_out[i] = (k >= G) ? 1 : 0;
        }
        return;
    }

    // 2. radix select, 8 bits per pass from the most significant digit.  Once
    //    the digit's bucket holds exactly the keys still needed, all of them are
    //    kept and the lower digits cannot change the selection: stop there and
    //    compare keys on the digits examined so far.
    if (tid == 0) { s_prefix = 0ull; s_kk = k; s_done = 0; }
    unsigned long long mask = 0ull;
    for (int shift = 56; shift >= 0; shift -= 8) {
        for (int i = tid; i < 256; i += kSelThreads) hist[i] = 0u;
        __syncthreads();
        const unsigned long long prefix = s_prefix;
        for (int i = tid; i < G; i += kSelThreads) {
            const unsigned long long u = (unsigned long long)__double_as_longlong(kv[i]);
            if ((u & mask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            // lane l owns digits 255-8l .. 248-8l, highest first
            unsigned c[8];
            unsigned tot = 0;
            for (int j = 0; j < 8; ++j) { c[j] = hist[255 - 8 * tid - j]; tot += c[j]; }
            unsigned inc = tot;
            for (int o = 1; o < 32; o <<= 1) {
                const unsigned t = __shfl_up_sync(0xffffffffu, inc, o);
                if (tid >= o) inc += t;
            }
            unsigned cum = inc - tot;  // keys with a higher digit than this lane's
            const unsigned kk = (unsigned)s_kk;
            if (cum < kk && kk <= cum + tot) {
                for (int j = 0; j < 8; ++j) {
                    if (cum + c[j] >= kk) {
                        const unsigned d = 255u - 8u * tid - j;
                        s_prefix = prefix | ((unsigned long long)d << shift);
                        s_kk = (int)(kk - cum);
                        if (c[j] == kk - cum) s_done = 1;
                        break;
                    }
                    cum += c[j];
                }
            }
        }
        mask |= 0xFFull << shift;
        __syncthreads();
        if (s_done) break;
    }
    // T: the k-th largest key on the examined digits (`mask`); take_eq: how
    // many keys equal to T there are kept (all of them after an early stop)
    const unsigned long long T = s_prefix;
    const int take_eq = s_kk;

    // 3. ordered compaction
    int run_out = 0, run_eq = 0;
    for (int base = 0; base < G; base += kSelThreads) {
        const int i = base + tid;
        const bool valid = i < G;
        const unsigned long long u = valid ? (unsigned long long)__double_as_longlong(kv[i]) & mask : 0ull;
        const bool gt = valid && u > T;
        const bool eq = valid && u == T;
        int eq_tot, take_tot;
        const int eq_before = block_excl_count(eq, warp_tot, &eq_tot);
        const bool take = gt || (eq && run_eq + eq_before < take_eq);
        const int pos = block_excl_count(take, warp_tot, &take_tot);
        if (take) out_idx[run_out + pos] = i;
        if (keep_out && valid) keep_out[i] = take ? 1 : 0;
        run_eq += eq_tot;
        run_out += take_tot;
    }
}

// Row (filter) selects: one block per layer of the batch.
__global__ void __launch_bounds__(kSelThreads) k_select_rows(const __grid_constant__ BatchArgs ba)
{
    pdl_wait();  // after the kernel before it in the stream (the filter keys)
    const BLayer& L = ba.L[blockIdx.x];
    if (!L.do_rows) return;
    select_block(L.fkeys, L.F, 1, L.k_filters, 1, 0, L.fkeys, L.keys_out, L.filt_idx, L.rkeep);
}

// Column-group selects: one block per layer of the batch.
__global__ void __launch_bounds__(kSelThreads) k_select_cols(const __grid_constant__ BatchArgs ba)
{
    pdl_wait();  // after the kernel before it in the stream (the column keys)
    const BLayer& L = ba.L[blockIdx.x];
    if (!L.do_cols) return;
    select_block(L.parts, L.G, L.taps, L.k_cols, L.R, L.K, L.ckeys, L.keys_out ? L.keys_out + L.F : nullptr,
                 L.col_idx, L.ckeep);
}

// Row-chunk count of the column-key pass of one layer: enough blocks to fill
// the GPU, with the partial sums bounded to 16384 doubles.
int column_parts(long long K, long long nrows)
{
    long long r = (304 + (K + 31) / 32 - 1) / ((K + 31) / 32);
    r = std::min(r, 16384 / std::max(K, 1ll));
    r = std::min(r, std::max(nrows / 32, 1ll));
    return (int)std::max(r, 1ll);
}

template <typename T>
sadmm_status run_project_batch(const ProjItem* items, int n, cudaStream_t s)
{
    BatchArgs ba;
    memset(&ba, 0, sizeof(ba));
    ba.n = n;
    int fk = 0, ck = 0, ka = 0;
    bool any_rows = false, any_cols = false;
    for (int l = 0; l < n; ++l) {
        const ProjItem& it = items[l];
        const Geometry& g = it.g;
        BLayer& L = ba.L[l];
        const int F = (int)g.f, K = (int)g.k;
        double* fkeys = reinterpret_cast<double*>(it.ws);
        L.W = it.W;
        L.U = it.U;
        L.filt_idx = it.filt_idx;
        L.col_idx = it.col_idx;
        L.keys_out = it.keys_out;
        L.fkeys = fkeys;
        L.ckeys = fkeys + round_up(F, 32);
        L.parts = L.ckeys + round_up(K, 32);
        L.rkeep = it.rkeep;
        L.ckeep = it.colkind == SADMM_COL_NONE ? nullptr : it.ckeep;
        L.F = F;
        L.K = K;
        L.taps = (it.colkind == SADMM_COL_CHANNEL) ? (int)g.taps : 1;
        L.G = (it.colkind == SADMM_COL_CHANNEL) ? (int)g.cg : K;
        L.k_filters = it.k_filters;
        L.k_cols = it.k_cols;
        // Keeping every group of a kind needs no keys: the top-G of G keys is
        // the whole ascending index list.  Unless the caller asked for the
        // keys, such lists (and keep flags) are written by the keep-all pass.
        L.rows_all = (it.k_filters == F) && !it.keys_out;
        L.cols_all = (it.colkind != SADMM_COL_NONE) && (it.k_cols == L.G) && !it.keys_out;
        L.do_rows = !L.rows_all;
        L.do_cols = it.colkind != SADMM_COL_NONE && !L.cols_all;
        const bool all_rows = (it.k_filters == F);
        L.krows = all_rows ? nullptr : it.filt_idx;
        L.nrows = all_rows ? F : it.k_filters;
        L.R = L.do_cols ? column_parts(K, L.nrows) : 0;
        L.cblocks = (K + 31) / 32;
        L.fk0 = fk;
        L.ck0 = ck;
        L.ka0 = ka;
        L.ka_n = std::max(L.rows_all ? F : 0, L.cols_all ? L.G : 0);
        L.rpb = K <= 1024 ? 8 : 1;
        fk += L.do_rows ? (F + L.rpb - 1) / L.rpb : 0;
        ck += L.do_cols ? L.cblocks * L.R : 0;
        ka += (L.ka_n + 255) / 256;
        any_rows = any_rows || L.do_rows;
        any_cols = any_cols || L.do_cols;
    }
    // Row keys (with the lists of the kinds kept whole), row selects, column
    // keys over the kept rows, column selects: one launch each for the whole
    // batch (the column keys read the kept-row lists, so they follow the row
    // selects).
    ba.fk_total = fk;
    if (fk + ka > 0) launch_pdl(k_filter_keys<T>, dim3(fk + ka), dim3(256), 0, s, ba);
    if (any_rows) launch_pdl(k_select_rows, dim3(n), dim3(kSelThreads), 0, s, ba);
    if (any_cols) {
        launch_pdl(k_column_keys<T>, dim3(ck), dim3(256), 0, s, ba);
        launch_pdl(k_select_cols, dim3(n), dim3(kSelThreads), 0, s, ba);
    }
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace

size_t project_workspace_bytes(const Geometry& g, int colkind)
{
    (void)colkind;
    // filter keys, column keys, and the partial column keys (at most 16384,
    // at least one row chunk of K)
    const long long parts = std::max(16384ll, round_up(g.k, 32));
    return (size_t)(round_up(g.f, 32) + round_up(g.k, 32) + parts) * sizeof(double) + 256;
}

sadmm_status launch_project_batch(const ProjItem* items, int n, int wdt, cudaStream_t s)
{
    if (n < 1 || n > kMaxBatch) return SADMM_EINVAL;
    if (wdt == SADMM_BF16) return run_project_batch<__nv_bfloat16>(items, n, s);
    return run_project_batch<float>(items, n, s);
}

sadmm_status launch_project(const Geometry& g, const void* W, const void* U, int wdt, int k_filters,
                            int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out,
                            void* ws, cudaStream_t s, uint8_t* rkeep, uint8_t* ckeep)
{
    ProjItem it;
    it.g = g;
    it.W = W;
    it.U = U;
    it.Z = nullptr;
    it.k_filters = k_filters;
    it.colkind = colkind;
    it.k_cols = k_cols;
    it.filt_idx = filt_idx;
    it.col_idx = col_idx;
    it.keys_out = keys_out;
    it.ws = ws;
    it.rkeep = rkeep;
    it.ckeep = ckeep;
    return launch_project_batch(&it, 1, wdt, s);
}

// ---------------------------------------------------------------------------
// Projection without caller-provided scratch.
//
// Some callers cannot hand this library a device workspace: a plugin or host
// framework that passes only its input and output tensors and owns every
// allocation itself, or a serving loop that must not allocate (or risk an
// out-of-memory failure) once it is running.  For them the keys live in one
// fixed device array compiled into the library instead.  The array is
// kNoAllocScratchBytes on every GPU that loads the library and stays there
// until the process exits.  All calls share it: nothing in it has to start at
// zero (every key is written before it is read), but two calls that run at the
// same time on the GPU (different streams, no ordering between them) overwrite
// each other's keys and give wrong index lists.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchBytes = SADMM_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;
// Per device, the array's address once looked up.  Atomic: host threads that
// make their first call on one device at the same time may both look it up
// (they find the same address); neither reads a half-written pointer.
std::atomic<void*> g_noalloc_ptr[kNoAllocMaxDevices];

// Device address of the array on the current device; looked up once per device
// (host code only sees a stand-in for the array, never its device address).
cudaError_t noalloc_scratch(void** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kNoAllocMaxDevices) return cudaErrorInvalidDevice;
    void* p = g_noalloc_ptr[dev].load(std::memory_order_acquire);
    if (!p) {
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return cudaSuccess;
}

}  // namespace
}  // namespace sadmm

extern "C" sadmm_status sadmm_project_groups_noalloc(const sadmm_conv_desc* d, const void* W, const void* U,
                                                     int wdt, int k_filters, int colkind, int k_cols,
                                                     int* filt_idx, int* col_idx, double* keys_out,
                                                     void* stream)
{
    using namespace sadmm;
    NvtxRange range("sadmm_project_groups_noalloc");
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    st = check_project_args(g, W, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out);
    if (st != SADMM_OK) return st;
    // the layer's keys must fit the fixed array
    if (project_workspace_bytes(g, colkind) > kNoAllocScratchBytes) return SADMM_EUNSUPPORTED;
    void* ws = nullptr;
    if (noalloc_scratch(&ws) != cudaSuccess) return SADMM_ECUDA;
    return launch_project(g, W, U, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out, ws,
                          static_cast<cudaStream_t>(stream));
}
