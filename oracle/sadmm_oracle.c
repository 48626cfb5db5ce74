/*
 * sadmm_oracle.c -- CPU oracle for the structured-pruned CONV forward path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path links, loads or
 * calls this file: only tests/, __graft_entry__.smoke() and bench.py's CPU
 * baseline use it.  It shares no code, header, table or helper with the CUDA
 * library; the descriptor is passed as a plain int array.
 *
 * Everything is fp64, plain loops, no blocking and no reordering beyond the
 * definitions below (StructADMM, arXiv 1807.11091):
 *
 *   Weight tensor W of a CONV layer, A filters x B channels x C x D taps
 *   (Sec. 3, "Structured Pruning Formulation"; OIDHW here, with a temporal tap
 *   extent KT for 3-D layers).  Lowered to a GEMM matrix with one row per
 *   filter and one column per (channel, kt, kh, kw) tap (Sec. 3, "Combination
 *   of structured sparsities"): row pruning = filter-wise sparsity, column
 *   pruning = channel-wise or shape-wise sparsity.
 *
 *   Euclidean projection onto a group-cardinality set (Sec. 4, solution of
 *   the second ADMM subproblem, Eq. 4 and the three paragraphs after it):
 *   compute O_g = ||V_g||_F^2 for every group g, keep the k groups with the
 *   largest O_g, zero the rest.  V = W (+U when the dual is given).
 *
 *   Convolution: y[n,f,o] = ReLU(b[f] + sum_{c,kt,kh,kw} W[f,c,kt,kh,kw] *
 *   x[n, g*Cg+c, ot*st-pt+kt, oh*sh-ph+kh, ow*sw-pw+kw]), x outside the input
 *   counts as zero, g = f / (F/groups).
 *
 * Each function names the definition it follows.
 */
#include <stdlib.h>
#include <string.h>

/* Descriptor layout (int[16]): n c t h w f groups kt kh kw st sh sw pt ph pw */
enum { D_N, D_C, D_T, D_H, D_W, D_F, D_G, D_KT, D_KH, D_KW, D_ST, D_SH, D_SW,
       D_PT, D_PH, D_PW, D_COUNT };

static long out_extent(long in, long k, long s, long p) { return (in + 2 * p - k) / s + 1; }

/* Filter-wise keys (Sec. 4, filter-wise projection): O_a = ||V[a,:,:,:]||_F^2,
 * summed in ascending element order.  V is [F][K] row-major. */
void oracle_filter_keys(int F, int K, const double* V, double* keys)
{
    for (int a = 0; a < F; ++a) {
        double s = 0.0;
        for (int k = 0; k < K; ++k) s += V[(long)a * K + k] * V[(long)a * K + k];
        keys[a] = s;
    }
}

/* Shape-wise keys (Sec. 4, shape-wise projection): O_{b,c,d} = ||V[:,b,c,d]||_F^2
 * over the rows a with rows[a] != 0 (all rows when rows == NULL), summed in
 * ascending filter order.  Column j of the [F][K] matrix is one (b,c,d). */
void oracle_shape_keys(int F, int K, const double* V, const unsigned char* rows, double* keys)
{
    for (int j = 0; j < K; ++j) {
        double s = 0.0;
        for (int a = 0; a < F; ++a) {
            if (rows && !rows[a]) continue;
            s += V[(long)a * K + j] * V[(long)a * K + j];
        }
        keys[j] = s;
    }
}

/* Channel-wise keys (Sec. 4, channel-wise projection): O_b = ||V[:,b,:,:]||_F^2
 * over the kept rows; channel b owns the `taps` consecutive columns
 * b*taps .. b*taps+taps-1.  Summed in ascending element (memory) order. */
void oracle_channel_keys(int F, int Cg, int taps, const double* V,
                         const unsigned char* rows, double* keys)
{
    long K = (long)Cg * taps;
    for (int b = 0; b < Cg; ++b) {
        double s = 0.0;
        for (int a = 0; a < F; ++a) {
            if (rows && !rows[a]) continue;
            for (int t = 0; t < taps; ++t) {
                double v = V[(long)a * K + (long)b * taps + t];
                s += v * v;
            }
        }
        keys[b] = s;
    }
}

typedef struct { double key; int idx; } keyed;

/* Larger key first; equal keys: lower index first. */
static int by_key_desc_idx_asc(const void* pa, const void* pb)
{
    const keyed* a = (const keyed*)pa;
    const keyed* b = (const keyed*)pb;
    if (a->key > b->key) return -1;
    if (a->key < b->key) return 1;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

static int by_int_asc(const void* pa, const void* pb)
{
    int a = *(const int*)pa, b = *(const int*)pb;
    return (a > b) - (a < b);
}

/* Keep the k largest keys (Sec. 4: "keep ... corresponding to the ... largest
 * values").  Ties go to the lower group index.  Writes the kept indices in
 * ascending order to out[0..k) and returns k, or -1 when k is out of range. */
int oracle_topk(int G, const double* keys, int k, int* out)
{
    if (k < 0 || k > G) return -1;
    keyed* t = (keyed*)malloc(sizeof(keyed) * (size_t)(G > 0 ? G : 1));
    if (!t) return -1;
    for (int i = 0; i < G; ++i) { t[i].key = keys[i]; t[i].idx = i; }
    qsort(t, (size_t)G, sizeof(keyed), by_key_desc_idx_asc);
    for (int i = 0; i < k; ++i) out[i] = t[i].idx;
    qsort(out, (size_t)k, sizeof(int), by_int_asc);
    free(t);
    return k;
}

/* Direct convolution over the full (masked) weight tensor, images n0..n1-1.
 * x: [N][C][T][H][W], Wm: [F][Cg][KT][KH][KW], bm: [F], y: [n1-n0][F][OT][OH][OW].
 * One plain loop per index; parallel over (n, f) only. */
void oracle_conv(const int* d, const double* x, const double* Wm, const double* bm,
                 int relu, int n0, int n1, double* y)
{
    const long C = d[D_C], T = d[D_T], H = d[D_H], W = d[D_W];
    const long F = d[D_F], G = d[D_G];
    const long KT = d[D_KT], KH = d[D_KH], KW = d[D_KW];
    const long ST = d[D_ST], SH = d[D_SH], SW = d[D_SW];
    const long PT = d[D_PT], PH = d[D_PH], PW = d[D_PW];
    const long Cg = C / G, Fg = F / G;
    const long OT = out_extent(T, KT, ST, PT);
    const long OH = out_extent(H, KH, SH, PH);
    const long OW = out_extent(W, KW, SW, PW);
    const long nimg = n1 - n0;

    #pragma omp parallel for collapse(2) schedule(dynamic, 1)
    for (long nn = 0; nn < nimg; ++nn) {
        for (long f = 0; f < F; ++f) {
            const long n = n0 + nn;
            const long g = f / Fg;
            for (long ot = 0; ot < OT; ++ot)
            for (long oh = 0; oh < OH; ++oh)
            for (long ow = 0; ow < OW; ++ow) {
                double s = 0.0;
                for (long c = 0; c < Cg; ++c)
                for (long kt = 0; kt < KT; ++kt)
                for (long kh = 0; kh < KH; ++kh)
                for (long kw = 0; kw < KW; ++kw) {
                    const long it = ot * ST - PT + kt;
                    const long ih = oh * SH - PH + kh;
                    const long iw = ow * SW - PW + kw;
                    if (it < 0 || it >= T || ih < 0 || ih >= H || iw < 0 || iw >= W) continue;
                    const double wv = Wm[(((f * Cg + c) * KT + kt) * KH + kh) * KW + kw];
                    const double xv = x[((((n * C) + g * Cg + c) * T + it) * H + ih) * W + iw];
                    s += wv * xv;
                }
                s += bm[f];
                if (relu && s < 0.0) s = 0.0;
                y[(((nn * F + f) * OT + ot) * OH + oh) * OW + ow] = s;
            }
        }
    }
}

int oracle_abi_version(void) { return 1; }
