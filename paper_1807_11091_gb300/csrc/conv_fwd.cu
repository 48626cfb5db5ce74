// conv_fwd.cu -- pruned CONV forward as an implicit GEMM on the sm_103a tensor
// cores (Sec. 3: after filter-wise (row) and channel-/shape-wise (column)
// pruning the layer is a smaller full GEMM).
//
//   D[m, i] = sum_{j < K'} A[m, j] * Wp[i, j]
//   A[m, j] = x[n, g*Cg + c_j, ot*st-pt+kt_j, oh*sh-ph+kh_j, ow*sw-pw+kw_j]
//
// m runs over output pixels (N*OT*OH*OW), i over the kept filters of conv group
// g, j over the kept (channel, tap) columns.  Pixels are the MMA M side (128 per
// tile, one TMEM lane each), kept filters the N side (bn <= 256 per tile), so a
// gathered pixel tile is reused by every kept filter of the tile.
//
// One persistent CTA per SM, warp-specialised (896 threads):
//   warp 0      TMA producer: 64-column x bn-row boxes of Wp (128-byte swizzle)
//   warp 1      TMEM allocator and MMA issuer (tcgen05.mma kind::f16, bf16 in,
//               fp32 accumulate, 128 x n x 16 per instruction)
//   warps 4-11  epilogue (two warps per TMEM lane quadrant): tcgen05.ld of the accumulator (lane = pixel), bias,
//               ReLU, coalesced stores to the NCHW output (consecutive lanes
//               write consecutive pixels of one filter plane), and zero-fill of
//               the pruned filters' planes for the tile's pixels
//   warps 12-27 gather, in two sets that fill alternate stages: in a set, each
//               thread builds two 16-byte K-major chunks of A for two pixels
//               of the tile (rows pp and pp + 64) through the gather table,
//               with zero fill outside the input, into the 128-byte-swizzled
//               stage buffer
// Shared-memory stages are guarded by mbarriers; the accumulator is double
// buffered in TMEM so the epilogue of one tile overlaps the MMAs of the next.
#include <cuda.h>
#include <string.h>

#include "common.cuh"
#include "conv_common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kBM = 128;           // pixels per tile
constexpr int kBK = 64;            // GEMM columns per stage
constexpr int kGatherWarps = 16;
constexpr int kEpiWarps = 8;
constexpr int kThreads = (4 + kEpiWarps + kGatherWarps) * 32;
constexpr int kGatherThreads = kGatherWarps * 32;
// The gather warps form kGatherSets independent sets; set i fills the stages
// whose running index is i modulo kGatherSets, so the load latency of one
// stage overlaps the loads of the next.
constexpr int kGatherSets = 2;
constexpr int kSetThreads = kGatherThreads / kGatherSets;
// A gather thread builds kPixPerThread pixel rows (pp, pp + kPixStride, ...) of
// kChunksPerThread 16-byte column chunks each.  More pixels per thread mean
// fewer reads of the (broadcast) gather table per element: a 16-byte shared
// load takes four wavefronts of the L1 data pipe whatever its addresses, and
// that pipe also carries the gather's global loads.
constexpr int kPixPerThread = 2;
constexpr int kPixStride = kBM / kPixPerThread;                         // 64 pixel slots
constexpr int kChunksPerThread = 8 * kPixStride / kSetThreads;          // 2 chunks of 8 columns
static_assert(kSetThreads % kPixStride == 0 && kChunksPerThread * kSetThreads == 8 * kPixStride,
              "a gather set must split a 128 x 64 stage evenly");
constexpr int kATileBytes = kBM * kBK * 2;  // 16 KB
constexpr int kMaxStages = 8;        // A stages (and B stages when B streams)
constexpr int kStreamStages = 4;     // stages when B streams with A
constexpr int kResidentStages = 6;   // A stages when the packed weights stay in shared memory
constexpr int kMaxGroups = 64;
constexpr int kTabCap = 512;       // kept-row entries of an epilogue table buffer
// Fixed shared-memory tail: epilogue tables [2][kTabCap] offsets and biases,
// per-group counts, barriers and the TMEM address.  The zero-plane table
// [2][zcap] follows it.
constexpr int kTailOffBias = 0;
constexpr int kTailCounts = kTailOffBias + 2 * 2 * kTabCap * 4;
constexpr int kTailBars = kTailCounts + 2 * kMaxGroups * 4;
constexpr int kTailZero = kTailBars + 512;
constexpr int kTailCutFlag = kTailBars + 448;  // stream-K flags [piece 0 (run end), piece 1 (run start)][looked, arrived]
static_assert((3 * kMaxStages + 7) * 8 + 8 <= 448, "barriers, TMEM address and abort flag end below the flags");
static_assert(448 + 4 * 4 <= 512, "four stream-K flags fit the barrier area");
constexpr int kSmemTail = kTailZero;


struct ConvArgs {
    const __nv_bfloat16* x;
    void* y;
    const float* bias;
    const uint2* gather;  // [k_pad] {channel/tap offset in x, tap bits}
    const int* rowmap;
    const int* zeromap;
    const int* counts;
    int* status;
    int M;            // N * plane (below 2^31)
    long long x_total, y_total;  // elements of x and y (the debug build's index checks)
    long long x_chw;  // elements per input image
    long long thw;    // elements per input channel
    int units;        // work items: m_tiles * groups * upairs * splits (below 2^31)
    FastDiv split_div, upairs_div, mtiles_div, plane_div, ohw_div, ow_div;
    int splits;       // K' splits per output tile (1: no split)
    int ksps;         // stages per split
    float* partial;   // [splits][groups * n_pad][m_pad] fp32 partial sums (splits > 1)
    int m_pad;        // m_tiles * 128
    int ncols_all;    // groups * n_pad
    int hw, W, H, T;
    int F, groups, Cg, Fg;
    int OW, OHW, plane;
    int st, sh, sw, pt, ph, pw;
    int KT, KH, KW;
    int nks;  // k_pad / 64
    int bn, n_tiles, n_pad;
    int nacc;      // filter tiles per unit (TMEM accumulators sharing one A tile)
    int upairs;    // units per (pixel tile, group): ceil(n_tiles / nacc)
    int acc_bufs;  // accumulator sets in TMEM (2: the epilogue overlaps the next unit's MMAs)
    int b_res;     // 1: a conv group's packed weights stay in shared memory for all its units
    int stages;
    int k_pad;
    int n_cols;          // K' (columns past it are padding)
    int split_mask;      // tap-mask encoding: 0 one bit per tap, 1 row bits + kw bits
    uint32_t full_mask;  // the mask of a pixel whose every tap is inside the input
    int tmem_stride;
    int tmem_cols;
    int zcap;  // zero-plane offsets per table buffer kept in shared memory
    int relu;
    // stream-K: CTA b takes stages [b*sk_len, (b+1)*sk_len) of the units'
    // stages laid end to end; sk_len >= nks, so a unit is cut at most once
    int sk_len;      // 0: work items are whole units (or K' splits)
    FastDiv nks_div;
    int* skcnt;      // arrival counter per cut: cut b-1 lies at the start of CTA b's run
    float* skpart;   // partial sums [cut][piece 0 | 1][sk_cols][128 pixels]
    int sk_cols;     // nacc * bn
};

// Work item w is split sp (stages ks0 .. ks1-1 of K') of unit w / splits; a
// unit covers filter tiles p*nacc .. p*nacc+nacc-1 of conv group g for pixel
// tile mt.  Groups are outermost, so a CTA (items w, w + grid, ...) stays in
// one conv group for long runs and rarely reloads resident weights.
SADMM_DEV void decode_unit(const ConvArgs& a, int w, int& p, int& g, int& mt, int& sp, int& ks0, int& ks1)
{
    const uint32_t u = fdiv((uint32_t)w, a.split_div);
    sp = w - (int)(u * a.split_div.d);
    ks0 = sp * a.ksps;
    ks1 = min(a.nks, ks0 + a.ksps);
    const uint32_t t = fdiv(u, a.upairs_div);
    p = (int)(u - t * a.upairs_div.d);
    const uint32_t gq = fdiv(t, a.mtiles_div);
    mt = (int)(t - gq * a.mtiles_div.d);
    g = (int)gq;
}

// The work items of this CTA in order: whole units u = blockIdx.x, + grid, ...
// (K' splits included); or, under stream-K, the pieces of its run of stages
// [b*sk_len, (b+1)*sk_len): the piece of the unit cut at the run's start, then
// the piece of the unit cut at its end, then the whole units between them.
// Both pieces of every cut unit thus come early in their CTAs' runs, so the
// second to arrive finishes the unit while later units are still being
// computed, not at the end of the kernel.
struct Work {
    int it, end;  // whole units (stream-K: stage bounds of the middle, unit-aligned)
    int phase;    // stream-K: 0 start piece next, 1 end piece next, 2 whole units
};

template <bool SK>
SADMM_DEV Work work_begin(const ConvArgs& a)
{
    Work w;
    if (SK) {
        const int s0 = blockIdx.x * a.sk_len;
        const int e0 = min(s0 + a.sk_len, a.units * a.nks);
        // sk_len >= nks: a run that starts inside a unit goes past that unit's end
        w.it = ((int)fdiv((uint32_t)(s0 + a.nks - 1), a.nks_div)) * a.nks;
        const int t0 = (int)fdiv((uint32_t)e0, a.nks_div) * a.nks;
        w.end = t0 >= w.it ? t0 : e0;
        w.phase = 0;
    } else {
        w.it = blockIdx.x;
        w.end = a.units;
        w.phase = 2;
    }
    return w;
}

// Next work item: its unit and stage range ks0 .. ks1-1; false at the end.
template <bool SK>
SADMM_DEV bool work_next(const ConvArgs& a, Work& w, int& p, int& g, int& mt, int& sp, int& ks0, int& ks1)
{
    if (SK) {
        int b = 0, e = 0;
        while (w.phase < 2 && b == e) {
            const int s0 = blockIdx.x * a.sk_len;
            if (w.phase++ == 0) {
                if (s0 < w.it) { b = s0; e = w.it; }  // the run starts inside a unit
            } else {
                const int e0 = min(s0 + a.sk_len, a.units * a.nks);
                if (e0 > w.end) { b = w.end; e = e0; }  // the run ends inside a unit
            }
        }
        if (b == e) {
            if (w.it >= w.end) return false;
            b = w.it;
            e = w.it + a.nks;
            w.it = e;
        }
        const int u = (int)fdiv((uint32_t)b, a.nks_div);
        decode_unit(a, u, p, g, mt, sp, ks0, ks1);  // one split: sp = 0
        ks0 = b - u * a.nks;
        ks1 = ks0 + (e - b);
        return true;
    }
    if (w.it >= w.end) return false;
    decode_unit(a, w.it, p, g, mt, sp, ks0, ks1);
    w.it += gridDim.x;
    return true;
}

// Tap-validity mask of one output pixel: the rule of tap_mask (common.cuh),
// written against the kernel arguments directly (a call through tap_mask costs
// this 72-register kernel a spill).  The valid range of each kernel coordinate
// is formed in closed form (bits_between) instead of testing every tap: the
// gather warps compute it for two pixels per tile, and on the pruned AlexNet
// layers the loops cost 5-7 % of the kernel's time.
SADMM_DEV uint32_t pixel_mask(const ConvArgs& a, int it0, int ih0, int iw0)
{
    const int t_lo = max(0, -it0), t_hi = min(a.KT, a.T - it0);
    const int h_lo = max(0, -ih0), h_hi = min(a.KH, a.H - ih0);
    const int w_lo = max(0, -iw0), w_hi = min(a.KW, a.W - iw0);
    const uint32_t cm = bits_between(w_lo, w_hi), hm = bits_between(h_lo, h_hi);
    if (a.split_mask) {
        uint32_t rm = 0;
        for (int kt = t_lo; kt < t_hi; ++kt) rm |= hm << (kt * a.KH);
        return rm | (cm << 16);
    }
    uint32_t m = 0;
    for (int kt = t_lo; kt < t_hi; ++kt)
        for (int kh = h_lo; kh < h_hi; ++kh) m |= cm << ((kt * a.KH + kh) * a.KW);
    return m;
}

// Branch-free conditional gather: the 16-bit element at p when no tap bit of
// `bits` is set in the pixel's inverted mask nM (~mask: the taps outside the
// input), else 0 (a predicated load).  Testing against zero lets the and and
// the compare fold into one logic operation that writes the predicate
// (measured 2-4 % faster than testing (mask & bits) == bits).
SADMM_DEV uint32_t ldg_u16_if(const unsigned short* p, uint32_t bits, uint32_t nM, const ConvArgs& a)
{
    if ((bits & nM) == 0 &&
        !dbg_in(p - reinterpret_cast<const unsigned short*>(a.x), a.x_total, a.status))
        return 0;  // debug build: an index outside x
    uint32_t v;
    asm("{\n\t.reg .pred q;\n\t.reg .b32 t;\n\t"
        "and.b32 t, %2, %3;\n\t"
        "setp.eq.b32 q, t, 0;\n\t"
        "mov.b32 %0, 0;\n\t"
        "@q ld.global.nc.u16 %0, [%1];\n\t}"
        : "=r"(v)
        : "l"(p), "r"(nM), "r"(bits));
    return v;
}

// SK: stream-K work items (a.sk_len > 0); a separate instantiation keeps the
// whole-tile loops free of the extra state.
template <bool OUT_BF16, bool SK>
__global__ void __launch_bounds__(kThreads, 1)
    k_conv_fwd(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ ConvArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = a.stages;
    const uint32_t b_bytes = (uint32_t)a.bn * 128u;      // one Wp box (bn rows x 64 columns)
    const uint32_t bstage = b_bytes * (uint32_t)a.nacc;  // a B stage holds nacc boxes
    uint8_t* sA = smem;
    uint8_t* sB = smem + (size_t)S * kATileBytes;
    // resident weights: the nks boxes of one conv group's filter tile
    uint2* s_table = reinterpret_cast<uint2*>(sB + (a.b_res ? (size_t)a.nks * b_bytes : (size_t)S * bstage));
    uint8_t* tail = reinterpret_cast<uint8_t*>(s_table + a.k_pad);  // 512-byte aligned
    int* s_eoff = reinterpret_cast<int*>(tail + kTailOffBias);                   // [2][kTabCap] plane offsets
    float* s_ebias = reinterpret_cast<float*>(tail + kTailOffBias) + 2 * kTabCap;  // [2][kTabCap] biases
    int* s_counts = reinterpret_cast<int*>(tail + kTailCounts);
    int* s_zoff = reinterpret_cast<int*>(tail + kTailZero);  // [2][zcap] zero-plane offsets
    volatile int* s_cut = reinterpret_cast<volatile int*>(tail + kTailCutFlag);
    uint64_t* bars = reinterpret_cast<uint64_t*>(tail + kTailBars);
    uint64_t* full_a = bars;
    uint64_t* full_b = bars + S;
    uint64_t* empty = bars + 2 * S;
    uint64_t* acc_full = bars + 3 * S;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* drain = acc_empty + 2;
    uint64_t* b_full = drain + 1;   // resident weights landed
    uint64_t* b_empty = drain + 2;  // every MMA on the resident weights completed
    uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(drain + 3);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full_a[s], kSetThreads / 32);  // one arrival per gather warp of a set
            mbar_init(&full_b[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < a.acc_bufs; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], kEpiWarps);  // one arrival per epilogue warp
        }
        mbar_init(drain, 1);
        mbar_init(b_full, 1);
        mbar_init(b_empty, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tmem_holder, (uint32_t)a.tmem_cols);
        tmem_relinquish();
    }
    // Nothing above reads global memory: it overlaps the previous kernel's tail.
    pdl_wait();
    pdl_trigger();
    for (int i = threadIdx.x; i < 2 * a.groups; i += blockDim.x) s_counts[i] = a.counts[i];
    {
        // the gather table is the same for every tile: keep it in shared memory
        const uint4* src = reinterpret_cast<const uint4*>(a.gather);
        uint4* dst = reinterpret_cast<uint4*>(s_table);
        for (int i = threadIdx.x; i < a.k_pad / 2; i += blockDim.x) dst[i] = __ldg(src + i);
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tmap);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_holder;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer (Wp)
        if (lane == 0 && a.b_res) {
            // One load of the unit's filter tile (all nks boxes) per change of
            // (group, filter tile), after the MMAs on the previous one retired.
            long long cur = -1;
            uint32_t e_ph = 0;
            int loads = 0;
            Work wk = work_begin<SK>(a);
            int p, g, sp, ks0, ks1, mt;
            while (work_next<SK>(a, wk, p, g, mt, sp, ks0, ks1)) {
                if (s_counts[2 * g] <= p * a.bn) continue;
                const long long key = (long long)g * a.upairs + p;
                if (key == cur) continue;
                if (loads > 0) {
                    if (!mbar_wait(b_empty, e_ph, abort_flag, a.status)) break;
                    e_ph ^= 1u;
                }
                mbar_arrive_expect_tx(b_full, b_bytes * (uint32_t)a.nks);
                const int row0 = g * a.n_pad + p * a.bn;
                for (int ks = 0; ks < a.nks; ++ks)
                    tma_load_2d(sB + (size_t)ks * b_bytes, &tmap, b_full, ks * kBK, row0);
                cur = key;
                ++loads;
            }
            // the last load has landed before the CTA retires
            if (loads > 0) {
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(b_full, (uint32_t)((loads - 1) & 1)) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        } else if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            uint32_t issued_parity[kMaxStages];
            uint32_t issued_mask = 0;
            bool ok = true;
            Work wk = work_begin<SK>(a);
            int p, g, sp, ks0, ks1, mt;
            while (ok && work_next<SK>(a, wk, p, g, mt, sp, ks0, ks1)) {
                const int nt0 = p * a.nacc;
                if (s_counts[2 * g] <= nt0 * a.bn) continue;
                int nbox = 0;  // filter tiles of this unit with kept rows
                for (int i = 0; i < a.nacc; ++i)
                    if (nt0 + i < a.n_tiles && s_counts[2 * g] > (nt0 + i) * a.bn) nbox = i + 1;
                const int row0 = g * a.n_pad + nt0 * a.bn;
                for (int ks = ks0; ks < ks1; ++ks) {
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) { ok = false; break; }
                    mbar_arrive_expect_tx(&full_b[s], b_bytes * (uint32_t)nbox);
                    for (int i = 0; i < nbox; ++i)
                        tma_load_2d(sB + (size_t)s * bstage + (size_t)i * b_bytes, &tmap, &full_b[s], ks * kBK,
                                    row0 + i * a.bn);
                    issued_parity[s] = ph;
                    issued_mask |= 1u << s;
                    if (++s == S) { s = 0; ph ^= 1u; }
                }
            }
            // Every box this thread issued has landed before the CTA retires
            // (normally already true: the MMA consumed them).
            for (int q = 0; q < S; ++q) {
                if (!(issued_mask & (1u << q))) continue;
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(&full_b[q], issued_parity[q]) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
        __syncwarp();  // the whole warp reaches the block barrier below together
    } else if (warp == 1) {
        // ------------------------------------------------------- MMA issuer
        // The whole warp runs the loop (warp-uniform descriptors); one elected
        // lane issues the MMAs and the commits that track them.
        {
            int s = 0;
            uint32_t ph = 0;
            int ab = 0;
            uint32_t acc_ph = 0;
            bool ok = true;
            long long cur = -1;    // (group, filter tile) of the resident weights
            uint32_t bf_ph = 0;
            const uint32_t sB0 = smem_u32(sB);
            Work wk = work_begin<SK>(a);
            int p, g, sp, ks0, ks1, mt;
            while (ok && work_next<SK>(a, wk, p, g, mt, sp, ks0, ks1)) {
                const int cnt = s_counts[2 * g] - p * a.nacc * a.bn;  // kept rows from the unit's first tile
                if (cnt <= 0) continue;
                if (a.b_res) {
                    const long long key = (long long)g * a.upairs + p;
                    if (key != cur) {
                        if (cur >= 0) mma_commit_elect(b_empty);  // the old weights are free once these MMAs finish
                        if (!mbar_wait_warp(b_full, bf_ph, abort_flag, a.status)) break;
                        bf_ph ^= 1u;
                        cur = key;
                    }
                }
                // one accumulator per filter tile with kept rows, N rounded up to 16
                const int rows1 = (a.nacc == 2 && p * 2 + 1 < a.n_tiles) ? min(a.bn, cnt - a.bn) : 0;
                const uint32_t idesc0 = idesc_bf16_f32(kBM, min(a.bn, (cnt + 15) & ~15));
                const uint32_t idesc1 = idesc_bf16_f32(kBM, min(a.bn, (max(rows1, 16) + 15) & ~15));
                const bool two = rows1 > 0;
                if (!mbar_wait_warp(&acc_empty[ab], acc_ph ^ 1u, abort_flag, a.status)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(ab * a.nacc * a.tmem_stride);
                for (int ks = ks0; ks < ks1; ++ks) {
                    if (!mbar_wait_warp(&full_a[s], ph, abort_flag, a.status) ||
                        (!a.b_res && !mbar_wait_warp(&full_b[s], ph, abort_flag, a.status))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + (size_t)s * kATileBytes);
                    const uint32_t b0 = sB0 + (a.b_res ? (uint32_t)ks * b_bytes : (uint32_t)s * bstage);
                    // The issuing thread is on the critical path: straight-line
                    // code, descriptors in registers.
                    if (!two) {
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk)
                            mma_bf16_ss_elect(d_tmem, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32),
                                        idesc0, (ks != ks0 || kk != 0) ? 1u : 0u);
                    } else {
                        const uint32_t d1 = d_tmem + (uint32_t)a.tmem_stride;
                        const uint32_t b1 = b0 + b_bytes;
#pragma unroll
                        for (int kk = 0; kk < kBK / 16; ++kk) {
                            const uint64_t adesc = sdesc_kmajor_sw128(a0 + kk * 32);
                            const uint32_t acc = (ks != ks0 || kk != 0) ? 1u : 0u;
                            mma_bf16_ss_elect(d_tmem, adesc, sdesc_kmajor_sw128(b0 + kk * 32), idesc0, acc);
                            mma_bf16_ss_elect(d1, adesc, sdesc_kmajor_sw128(b1 + kk * 32), idesc1, acc);
                        }
                    }
                    mma_commit_elect(&empty[s]);
                    if (++s == S) { s = 0; ph ^= 1u; }
                }
                if (!ok) break;
                mma_commit_elect(&acc_full[ab]);
                if (++ab == a.acc_bufs) { ab = 0; acc_ph ^= 1u; }
            }
            // Every MMA this thread issued has completed before TMEM is freed.
            mma_commit_elect(drain);
            if (lane == 0) {
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(drain, 0) && globaltimer() - t0 < kWaitLimitNs) {}
            }
        }
        __syncwarp();
    } else if (warp >= 4 && warp < 4 + kEpiWarps) {
        // --------------------------------------------------------- epilogue
        // kEpiWarps / 4 warps share each TMEM lane quadrant and take its
        // 16-column chunks in turn, then the zero planes.  The output-plane
        // offset and bias of every packed row, and the offsets of the pruned
        // filters' planes, sit in shared memory; they are reloaded only when
        // a unit's (conv group, filter tiles) differ from the previous one's.
        constexpr int kHalves = kEpiWarps / 4;
        const int q = warp & 3;  // TMEM lane quadrant this warp may access
        const int h = (warp - 4) >> 2;
        const int et = threadIdx.x - 4 * 32;  // 0 .. kEpiWarps*32-1
        const int row = q * 32 + lane;
        int ab = 0;
        uint32_t acc_ph = 0;
        int ub = 1;         // table buffer of the current unit
        long long tab_key = -1;  // (group, filter tiles) the tables hold
        // After a failed wait (another role aborted) the warp keeps walking the
        // units, without TMEM or stores, so the named barrier stays balanced.
        bool alive = true;
        Work wk = work_begin<SK>(a);
        int p, g, sp, ks0, ks1, mt;
        while (work_next<SK>(a, wk, p, g, mt, sp, ks0, ks1)) {
            const int nt0 = p * a.nacc;
            const int cnt = s_counts[2 * g] - nt0 * a.bn;  // kept rows from the unit's first tile
            const int zc = (p == 0) ? s_counts[2 * g + 1] : 0;  // pruned filters whose planes this unit zeroes
            const long long key = (long long)g * a.upairs + p;
            if (key != tab_key) {
                ub ^= 1;
                int* u_off = s_eoff + ub * kTabCap;
                float* u_bias = s_ebias + ub * kTabCap;
                if (cnt > 0) {
                    // column i of the unit = row i % bn of filter tile nt0 + i / bn
                    const int* rmap = a.rowmap + (long long)g * a.n_pad + (long long)nt0 * a.bn;
                    const int ncol = min(a.nacc, a.n_tiles - nt0) * a.bn;
                    for (int i = et; i < ncol; i += kEpiWarps * 32) {
                        const int f = __ldg(rmap + i);
                        u_off[i] = f >= 0 ? f * a.plane : 0;
                        u_bias[i] = (f >= 0 && a.bias) ? __ldg(a.bias + f) : 0.0f;
                    }
                }
                const int* zmap = a.zeromap + (long long)g * a.Fg;
                int* u_zero = s_zoff + ub * a.zcap;
                for (int i = et; i < min(zc, a.zcap); i += kEpiWarps * 32) u_zero[i] = __ldg(zmap + i) * a.plane;
                asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
                tab_key = key;
            }
            const int* u_off = s_eoff + ub * kTabCap;
            const float* u_bias = s_ebias + ub * kTabCap;
            // stream-K: a unit cut at the start of CTA b's run has piece 0 (its
            // first stages) in CTA b-1 and piece 1 in CTA b, and cut index b-1
            const bool cut = SK && (ks0 > 0 || ks1 < a.nks);
            const int piece = ks0 > 0 ? 1 : 0;
            const int cut_idx = (int)blockIdx.x - piece;
            const int m = mt * kBM + row;
            const bool valid = m < a.M;
            const long long n_img = valid ? (long long)fdiv((uint32_t)m, a.plane_div) : 0;
            const long long pix = valid ? m - n_img * a.plane : 0;
            float* yf = reinterpret_cast<float*>(a.y) + (n_img * (long long)a.F * a.plane + pix);
            __nv_bfloat16* yh = reinterpret_cast<__nv_bfloat16*>(a.y) + (n_img * (long long)a.F * a.plane + pix);
            const YCheck yc{n_img * (long long)a.F * a.plane + pix, a.y_total, a.status};
            int chunks = 0;  // chunks of this unit so far (zero planes, then accumulator columns)
            if (zc > 0 && alive && a.splits == 1 && ks0 == 0) {
                // Pruned filters of this conv group: their planes are zero.  They
                // need no accumulator, so they go out while the unit's MMAs run;
                // these chunks of 16 planes start the unit's chunk sequence
                // (warp-uniform: it decides which warp reads which TMEM chunk).
                const int* zmap = a.zeromap + (long long)g * a.Fg;
                const int* u_zero = s_zoff + ub * a.zcap;
                const int nzc = (zc + kEpiCols - 1) / kEpiCols;
                for (int k = h; valid && k < nzc; k += kHalves) {
                    const int z0 = k * kEpiCols;
                    if (z0 + kEpiCols <= a.zcap && z0 + kEpiCols <= zc) {
#pragma unroll
                        for (int j = 0; j < kEpiCols; j += 4) {
                            const int4 o = *reinterpret_cast<const int4*>(u_zero + z0 + j);
                            if (!(y_ok(yc, o.x) && y_ok(yc, o.y) && y_ok(yc, o.z) && y_ok(yc, o.w))) continue;
                            if (OUT_BF16) {
                                const __nv_bfloat16 zb = __float2bfloat16_rn(0.0f);
                                yh[o.x] = zb; yh[o.y] = zb; yh[o.z] = zb; yh[o.w] = zb;
                            } else {
                                __stcs(yf + o.x, 0.0f); __stcs(yf + o.y, 0.0f);
                                __stcs(yf + o.z, 0.0f); __stcs(yf + o.w, 0.0f);
                            }
                        }
                    } else {
                        for (int z = z0; z < min(z0 + kEpiCols, zc); ++z) {
                            const int off = z < a.zcap ? u_zero[z] : __ldg(zmap + z) * a.plane;
                            if (!y_ok(yc, off)) continue;
                            if (OUT_BF16)
                                yh[off] = __float2bfloat16_rn(0.0f);
                            else
                                __stcs(yf + off, 0.0f);
                        }
                    }
                }
                chunks = nzc;
            }
            // warp-uniform outcome: the TMEM loads below are .sync.aligned
            if (cnt > 0 && alive && !__all_sync(0xffffffffu, mbar_wait(&acc_full[ab], acc_ph, abort_flag, a.status)))
                alive = false;
            // Stream-K piece of a cut unit.  If the unit's other piece has
            // arrived already, this one finishes the unit: its accumulator plus
            // the other's fp32 partial sums, then bias, ReLU, stores (mode 2).
            // Otherwise it writes its own partial sums and arrives (mode 1);
            // should the other piece have arrived meanwhile, it finishes after
            // all.  The two-term fp32 sum is the same whichever piece adds it.
            int cut_mode = 0;
            volatile int* cf = s_cut + 2 * piece;  // [looked, arrived]: one pair per head / tail piece of the CTA
            const float* other = nullptr;
            if (cut && cnt > 0) {
                if (et == 0) {
                    const int seen = alive ? ld_acquire_gpu(a.skcnt + cut_idx) : 0;
                    if (seen) st_relaxed_gpu(a.skcnt + cut_idx, 0);  // zero again for the next launch
                    cf[0] = seen;
                }
                asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
                cut_mode = cf[0] ? 2 : 1;
                other = a.skpart + (size_t)(cut_idx * 2 + 1 - piece) * a.sk_cols * kBM + row;
            }
            if (cnt > 0 && alive) {
                tc_fence_after();
                for (int ti = 0; ti < a.nacc && nt0 + ti < a.n_tiles; ++ti) {
                    const int nrows = min(a.bn, cnt - ti * a.bn);
                    if (nrows <= 0) break;
                    const int nch = (nrows + kEpiCols - 1) / kEpiCols;
                    const uint32_t taddr = tmem_base + (uint32_t)((ab * a.nacc + ti) * a.tmem_stride) +
                                           ((uint32_t)(q * 32) << 16);
                    const int* t_off = u_off + ti * a.bn;
                    const float* t_bias = u_bias + ti * a.bn;
                    // chunk k of this tile is the unit's chunk chunks + k; warp h takes those = h mod kHalves
                    for (int k = (h - chunks % kHalves + kHalves) % kHalves; k < nch; k += kHalves) {
                        const int c0 = k * kEpiCols;
                        uint32_t r[kEpiCols];
                        tmem_ld_32x32b_x16(taddr + (uint32_t)c0, r);
                        tmem_ld_wait();
                        const size_t col0 = ((size_t)ti * a.bn + c0) * kBM;  // partial-sum offset of the chunk
                        if (cut_mode == 1) {
                            // this piece's raw fp32 partial sums, every lane (pixel) of the tile
                            float* pp = a.skpart + (size_t)(cut_idx * 2 + piece) * a.sk_cols * kBM + row + col0;
#pragma unroll
                            for (int j = 0; j < kEpiCols; ++j) __stcg(pp + (size_t)j * kBM, __uint_as_float(r[j]));
                        } else if (cut_mode == 2) {
                            float v[kEpiCols];
#pragma unroll
                            for (int j = 0; j < kEpiCols; ++j)
                                v[j] = __uint_as_float(r[j]) + __ldcg(other + col0 + (size_t)j * kBM);
                            if (valid) store_cols<OUT_BF16>(v, c0, nrows, t_off, t_bias, a.relu, yf, yh, yc);
                        } else if (valid && a.splits > 1) {
                            // split K': raw fp32 partial sums, [split][column][pixel]
                            float* pp = a.partial +
                                        ((size_t)sp * a.ncols_all + (size_t)g * a.n_pad + (size_t)(nt0 + ti) * a.bn + c0) *
                                            a.m_pad +
                                        m;
#pragma unroll
                            for (int j = 0; j < kEpiCols; ++j)
                                if (c0 + j < nrows) __stcs(pp + (size_t)j * a.m_pad, __uint_as_float(r[j]));
                        } else if (valid) {
                            float v[kEpiCols];
#pragma unroll
                            for (int j = 0; j < kEpiCols; ++j) v[j] = __uint_as_float(r[j]);
                            store_cols<OUT_BF16>(v, c0, nrows, t_off, t_bias, a.relu, yf, yh, yc);
                        }
                    }
                    chunks += nch;
                }
            }
            if (cut_mode == 1) {
                // every partial store of this CTA's epilogue precedes the arrival
                asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
                if (et == 0) {
                    int last = 0;
                    if (alive) {
                        last = atom_add_acq_rel_gpu(a.skcnt + cut_idx, 1) == 1;
                        if (last) st_relaxed_gpu(a.skcnt + cut_idx, 0);
                    }
                    cf[1] = last;
                }
                asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
                if (cf[1] && alive) {
                    // the other piece arrived first after all: finish from TMEM
                    int ch = 0;
                    for (int ti = 0; ti < a.nacc && nt0 + ti < a.n_tiles; ++ti) {
                        const int nrows = min(a.bn, cnt - ti * a.bn);
                        if (nrows <= 0) break;
                        const int nch = (nrows + kEpiCols - 1) / kEpiCols;
                        const uint32_t taddr = tmem_base + (uint32_t)((ab * a.nacc + ti) * a.tmem_stride) +
                                               ((uint32_t)(q * 32) << 16);
                        const int* t_off = u_off + ti * a.bn;
                        const float* t_bias = u_bias + ti * a.bn;
                        for (int k = (h - ch % kHalves + kHalves) % kHalves; k < nch; k += kHalves) {
                            const int c0 = k * kEpiCols;
                            uint32_t r[kEpiCols];
                            tmem_ld_32x32b_x16(taddr + (uint32_t)c0, r);
                            tmem_ld_wait();
                            const size_t col0 = ((size_t)ti * a.bn + c0) * kBM;
                            float v[kEpiCols];
#pragma unroll
                            for (int j = 0; j < kEpiCols; ++j)
                                v[j] = __uint_as_float(r[j]) + __ldcg(other + col0 + (size_t)j * kBM);
                            if (valid) store_cols<OUT_BF16>(v, c0, nrows, t_off, t_bias, a.relu, yf, yh, yc);
                        }
                        ch += nch;
                    }
                }
            }
            if (cnt > 0 && alive) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_empty[ab]);
                if (++ab == a.acc_bufs) { ab = 0; acc_ph ^= 1u; }
            }
        }
    } else if (warp >= 4 + kEpiWarps) {
        // ----------------------------------------------------------- gather
        const int gt = threadIdx.x - (4 + kEpiWarps) * 32;
        const int set = gt / kSetThreads;
        const int st = gt - set * kSetThreads;
        const int pp = st % kPixStride;                        // first pixel row of this thread
        const int chunk0 = (st / kPixStride) * kChunksPerThread;  // its chunks chunk0 .. + kChunksPerThread - 1
        const unsigned short* xs = reinterpret_cast<const unsigned short*>(a.x);
        int s = 0;
        uint32_t ph = 0;
        int turn = 0;  // running stage index modulo kGatherSets
        bool ok = true;
        Work wk = work_begin<SK>(a);
        int p, g, sp, ks0, ks1, mt;
        while (ok && work_next<SK>(a, wk, p, g, mt, sp, ks0, ks1)) {
            if (s_counts[2 * g] <= p * a.nacc * a.bn) continue;
            uint32_t M[kPixPerThread];
            const unsigned short* xb[kPixPerThread];
            bool full = true;
#pragma unroll
            for (int r = 0; r < kPixPerThread; ++r) {
                const int m = mt * kBM + pp + r * kPixStride;
                M[r] = 0;
                xb[r] = xs;
                if (m < a.M) {
                    const long long n_img = fdiv((uint32_t)m, a.plane_div);
                    const int pix = (int)(m - n_img * a.plane);
                    const int ot = (int)fdiv((uint32_t)pix, a.ohw_div);
                    const int r2 = pix - ot * a.OHW;
                    const int oh = (int)fdiv((uint32_t)r2, a.ow_div);
                    const int ow = r2 - oh * a.OW;
                    const int it0 = ot * a.st - a.pt, ih0 = oh * a.sh - a.ph, iw0 = ow * a.sw - a.pw;
                    M[r] = pixel_mask(a, it0, ih0, iw0);
                    xb[r] = xs + (n_img * a.x_chw + (long long)g * a.Cg * a.thw + (long long)it0 * a.hw +
                                  (long long)ih0 * a.W + iw0);
                }
                full = full && M[r] == a.full_mask;
                M[r] = ~M[r];  // the predicated loads test the taps outside the input
            }
            // Every lane's pixels see every tap: no bounds test is needed.
            const bool interior = __all_sync(0xffffffffu, full);
            for (int ks = ks0; ks < ks1; ++ks) {
                if (turn == set) {
                    // Issue every load of this thread's columns first (they
                    // read only x), then wait for the stage buffer and store.
                    const uint2* te = s_table + (size_t)ks * kBK;
                    uint32_t v[8 * kChunksPerThread * kPixPerThread];  // [pixel][chunk][column]
                    // two table entries per 16-byte shared-memory load, used for every pixel of the thread
                    const uint4* te4 = reinterpret_cast<const uint4*>(te);
                    if (interior && (ks + 1) * kBK <= a.n_cols) {
#pragma unroll
                        for (int ci = 0; ci < kChunksPerThread; ++ci) {
#pragma unroll
                            for (int e = 0; e < 8; e += 2) {
                                const uint4 t = te4[((chunk0 + ci) * 8 + e) >> 1];
#pragma unroll
                                for (int r = 0; r < kPixPerThread; ++r) {
                                    v[(r * kChunksPerThread + ci) * 8 + e] =
                                        dbg_in(xb[r] + (int)t.x - xs, a.x_total, a.status) ? __ldg(xb[r] + (int)t.x) : 0u;
                                    v[(r * kChunksPerThread + ci) * 8 + e + 1] =
                                        dbg_in(xb[r] + (int)t.z - xs, a.x_total, a.status) ? __ldg(xb[r] + (int)t.z) : 0u;
                                }
                            }
                        }
                    } else {
#pragma unroll
                        for (int ci = 0; ci < kChunksPerThread; ++ci) {
#pragma unroll
                            for (int e = 0; e < 8; e += 2) {
                                const uint4 t = te4[((chunk0 + ci) * 8 + e) >> 1];
#pragma unroll
                                for (int r = 0; r < kPixPerThread; ++r) {
                                    v[(r * kChunksPerThread + ci) * 8 + e] = ldg_u16_if(xb[r] + (int)t.x, t.y, M[r], a);
                                    v[(r * kChunksPerThread + ci) * 8 + e + 1] =
                                        ldg_u16_if(xb[r] + (int)t.z, t.w, M[r], a);
                                }
                            }
                        }
                    }
                    if (!mbar_wait(&empty[s], ph ^ 1u, abort_flag, a.status)) { ok = false; break; }
                    uint8_t* tile = sA + (size_t)s * kATileBytes;
#pragma unroll
                    for (int r = 0; r < kPixPerThread; ++r) {
#pragma unroll
                        for (int ci = 0; ci < kChunksPerThread; ++ci) {
                            const uint32_t* q = v + (r * kChunksPerThread + ci) * 8;
                            *reinterpret_cast<uint4*>(
                                tile + sw128_offset((uint32_t)(pp + r * kPixStride), (uint32_t)(chunk0 + ci))) =
                                make_uint4(__byte_perm(q[0], q[1], 0x5410), __byte_perm(q[2], q[3], 0x5410),
                                           __byte_perm(q[4], q[5], 0x5410), __byte_perm(q[6], q[7], 0x5410));
                        }
                    }
                // every lane's stores are visible to the tensor core's async
                    // proxy, then one arrival for the warp
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&full_a[s]);
                }
                if (++s == S) { s = 0; ph ^= 1u; }
                if (++turn == kGatherSets) turn = 0;
            }
        }
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, (uint32_t)a.tmem_cols);
    }
}

// Split K': y = ReLU(bias + sum of the splits' partial sums, in split order)
// for every kept row, zeros for the pruned filters' planes.  Block (bx, r):
// row r of [kept rows of all groups | pruned-filter slots], pixels
// bx*1024 .. bx*1024+1023.
template <bool OUT_BF16>
__global__ void __launch_bounds__(256) k_splitk_finalize(const ConvArgs a)
{
    pdl_wait();  // the partial sums of the conv kernel before it
    const int r = blockIdx.y;
    int f;
    bool zero;
    if (r < a.ncols_all) {
        f = __ldg(a.rowmap + r);
        zero = false;
    } else {
        const int z = r - a.ncols_all;
        const int g = z / a.Fg, zi = z - g * a.Fg;
        if (zi >= __ldg(a.counts + 2 * g + 1)) return;
        f = __ldg(a.zeromap + g * a.Fg + zi);
        zero = true;
    }
    if (f < 0) return;
    const float b = (!zero && a.bias) ? __ldg(a.bias + f) : 0.0f;
    for (int q = 0; q < 4; ++q) {
        const int m = blockIdx.x * 1024 + q * 256 + threadIdx.x;
        if (m >= a.M) break;
        float v = 0.0f;
        if (!zero) {
            float acc = 0.0f;
            for (int sp = 0; sp < a.splits; ++sp)
                acc += __ldcs(a.partial + ((size_t)sp * a.ncols_all + r) * a.m_pad + m);
            v = acc + b;
            if (a.relu) v = fmaxf(v, 0.0f);
        }
        const int n_img = (int)fdiv((uint32_t)m, a.plane_div);
        const size_t off = ((size_t)n_img * a.F + f) * a.plane + (m - n_img * a.plane);
        if (!dbg_in((long long)off, a.y_total, a.status)) continue;
        if (OUT_BF16)
            reinterpret_cast<__nv_bfloat16*>(a.y)[off] = __float2bfloat16_rn(v);
        else
            reinterpret_cast<float*>(a.y)[off] = v;
    }
}

template <bool OUT_BF16, bool SK>
cudaError_t launch(const CUtensorMap& map, const ConvArgs& a, int grid, size_t smem, cudaStream_t s)
{
    auto kern = k_conv_fwd<OUT_BF16, SK>;
    static int configured_dev = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_dev != dev) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
        if (e != cudaSuccess) return e;
        configured_dev = dev;
    }
    // Both kernels may be scheduled while the kernel before them finishes
    // (programmatic dependent launch); each waits for it before reading memory.
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, map, a);
    if (e != cudaSuccess) return e;
    if (a.splits > 1) {
        cfg.gridDim = dim3((unsigned)((a.M + 1023) / 1024), (unsigned)(a.ncols_all + a.groups * a.Fg));
        cfg.blockDim = dim3(256);
        cfg.dynamicSmemBytes = 0;
        e = cudaLaunchKernelEx(&cfg, k_splitk_finalize<OUT_BF16>, a);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

}  // namespace

sadmm_status launch_conv_fwd(const sadmm_plan* plan, const Geometry& g, const void* x, const float* bias,
                             int relu, void* y, int ydt, int phase, cudaStream_t s)
{
    if (plan->xs_mode) return launch_conv_slab(plan, g, x, bias, relu, y, ydt, phase, s);
    if (phase == SADMM_FWD_INPUT) return SADMM_OK;  // the gathered path reads x in its own kernel
    if (g.groups > kMaxGroups) return SADMM_EUNSUPPORTED;
    const char* base = static_cast<const char*>(plan->dev);
    ConvArgs a;
    memset(&a, 0, sizeof(a));
    a.x = static_cast<const __nv_bfloat16*>(x);
    a.y = y;
    a.bias = bias;
    a.gather = reinterpret_cast<const uint2*>(base + plan->off_gather);
    a.rowmap = reinterpret_cast<const int*>(base + plan->off_rowmap);
    a.zeromap = reinterpret_cast<const int*>(base + plan->off_zeromap);
    a.counts = reinterpret_cast<const int*>(base + plan->off_counts);
    a.status = device_status_ptr();
    if (g.m >= (1ll << 31) - 256) return SADMM_EUNSUPPORTED;  // pixel indices stay in int
    a.M = (int)g.m;
    a.x_total = g.n * g.c * g.t * g.h * g.w;
    a.y_total = g.n * g.f * g.plane;
    a.x_chw = g.c * g.t * g.h * g.w;
    a.thw = g.t * g.h * g.w;
    a.hw = (int)(g.h * g.w);
    a.W = (int)g.w;
    a.H = (int)g.h;
    a.T = (int)g.t;
    a.F = (int)g.f;
    a.groups = (int)g.groups;
    a.Cg = (int)g.cg;
    a.Fg = (int)g.fg;
    a.OW = (int)g.ow;
    a.OHW = (int)(g.oh * g.ow);
    a.plane = (int)g.plane;
    a.st = (int)g.st;
    a.sh = (int)g.sh;
    a.sw = (int)g.sw;
    a.pt = (int)g.pt;
    a.ph = (int)g.ph;
    a.pw = (int)g.pw;
    a.KT = (int)g.kt;
    a.KH = (int)g.kh;
    a.KW = (int)g.kw;
    a.nks = plan->k_pad / kBK;
    a.bn = plan->bn;
    a.n_tiles = plan->n_tiles;
    a.nacc = plan->n_tiles >= 2 ? 2 : 1;
    a.upairs = (plan->n_tiles + a.nacc - 1) / a.nacc;
    a.n_pad = plan->n_pad;
    a.relu = relu ? 1 : 0;
    const long long m_tiles = (g.m + kBM - 1) / kBM;
    a.splits = plan->splits > 1 ? plan->splits : 1;
    a.ksps = a.splits > 1 ? plan->stages_per_split : a.nks;
    if (a.splits > 1 && ((long long)a.ksps * (a.splits - 1) >= a.nks || (long long)a.ksps * a.splits < a.nks))
        return SADMM_EINVAL;  // a plan whose split does not tile K'
    a.partial = a.splits > 1 ? reinterpret_cast<float*>(const_cast<char*>(base) + plan->off_partial) : nullptr;
    a.m_pad = (int)(m_tiles * kBM);
    a.ncols_all = (int)(g.groups * plan->n_pad);
    a.split_div = make_fastdiv((uint32_t)a.splits);
    const long long units = m_tiles * g.groups * a.upairs * a.splits;
    if (units >= (1ll << 31) - (1ll << 20)) return SADMM_EUNSUPPORTED;  // u + grid stays below 2^31
    a.units = (int)units;
    a.upairs_div = make_fastdiv((uint32_t)a.upairs);
    a.mtiles_div = make_fastdiv((uint32_t)m_tiles);
    a.plane_div = make_fastdiv((uint32_t)g.plane);
    a.ohw_div = make_fastdiv((uint32_t)(g.oh * g.ow));
    a.ow_div = make_fastdiv((uint32_t)g.ow);

    a.k_pad = plan->k_pad;
    a.n_cols = plan->n_cols;
    a.split_mask = tap_mask_mode(g);
    if (a.split_mask)
        a.full_mask = ((1u << (g.kt * g.kh)) - 1u) | (((1u << g.kw) - 1u) << 16);
    else
        a.full_mask = (uint32_t)((1ull << g.taps) - 1ull);
    const int table_bytes = plan->k_pad * 8;
    const int budget = 232448 - 1024 - kSmemTail - table_bytes;
    // One filter tile per group: keep the group's packed weights (nks boxes)
    // in shared memory when that leaves room for at least 3 A stages.
    const long long res_bytes = (long long)plan->bn * 128 * a.nks;
    int stage_bytes;
    long long fixed_bytes;
    // (not when K' is split: a work item then uses only a few of the boxes)
    if (plan->n_tiles == 1 && plan->splits <= 1 && budget - res_bytes >= 3LL * kATileBytes) {
        a.b_res = 1;
        stage_bytes = kATileBytes;
        fixed_bytes = res_bytes;
        a.stages = (int)((budget - res_bytes) / kATileBytes);
        if (a.stages > kResidentStages) a.stages = kResidentStages;
    } else {
        // At most kStreamStages: what shared memory leaves over serves as L1 for x.
        a.b_res = 0;
        stage_bytes = kATileBytes + a.nacc * plan->bn * 128;
        fixed_bytes = 0;
        a.stages = budget / stage_bytes;
        if (a.stages > kStreamStages) a.stages = kStreamStages;
        if (a.stages < 2) return SADMM_EUNSUPPORTED;
    }
    // Zero-plane offsets of a conv group (at most min(Fg, F - kept)) in shared
    // memory, as far as the stages leave room; the rest are read from HBM.
    {
        long long zmax = g.f - plan->n_filt;
        if (zmax > g.fg) zmax = g.fg;
        if (zmax < 0) zmax = 0;
        long long room = (budget - fixed_bytes - (long long)a.stages * stage_bytes) / 8;  // two buffers of 4-byte entries
        if (room > 4096) room = 4096;
        a.zcap = (int)(((zmax < room ? zmax : room) + 3) & ~3LL);
        if ((long long)a.zcap > room) a.zcap = (int)(room & ~3LL);
    }
    a.tmem_stride = (plan->bn + 31) & ~31;
    a.acc_bufs = (2 * a.nacc * a.tmem_stride <= 512) ? 2 : 1;
    int cols = 32;
    while (cols < a.acc_bufs * a.nacc * a.tmem_stride) cols <<= 1;
    a.tmem_cols = cols;
    const size_t smem =
        1024 + (size_t)fixed_bytes + (size_t)a.stages * stage_bytes + table_bytes + kSmemTail + (size_t)a.zcap * 8;

    long long grid = plan->ctas > 0 ? plan->ctas : device_sm_count();
    if (grid > a.units) grid = a.units;
    if (grid < 1) grid = 1;
    if (plan->sk_len > 0) {
        // stream-K: the plan's run length and CTA count must tile the stages
        // with every unit cut at most once
        const long long total = units * a.nks;
        const long long L = plan->sk_len;
        if (a.splits > 1 || L < a.nks || total >= (1ll << 31) - (1ll << 20) || plan->sk_grid != (total + L - 1) / L ||
            a.acc_bufs != 2)
            return SADMM_EINVAL;
        a.sk_len = (int)L;
        a.nks_div = make_fastdiv((uint32_t)a.nks);
        a.sk_cols = a.nacc * plan->bn;
        a.skcnt = reinterpret_cast<int*>(const_cast<char*>(base) + plan->off_sk);
        a.skpart = reinterpret_cast<float*>(const_cast<char*>(base) + plan->off_sk +
                                            round_up((long long)plan->sk_grid * 4, 1024));
        grid = plan->sk_grid;
    }

    CUtensorMap map;
    memcpy(&map, plan->tmap, sizeof(map));
    cudaError_t e;
    if (a.sk_len > 0)
        e = (ydt == SADMM_BF16) ? launch<true, true>(map, a, (int)grid, smem, s)
                                : launch<false, true>(map, a, (int)grid, smem, s);
    else
        e = (ydt == SADMM_BF16) ? launch<true, false>(map, a, (int)grid, smem, s)
                                : launch<false, false>(map, a, (int)grid, smem, s);
    return e == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace sadmm
