/*
 * sadmm.h -- C ABI of libsadmm: the forward pass of a CONV layer whose weights
 * are structurally pruned (StructADMM, arXiv 1807.11091), on one sm_103a GPU.
 *
 * Three calls make up the path, in the paper's order:
 *
 *   sadmm_project_groups  Euclidean projection of V = W (+U) onto a structured
 *                         sparsity set: squared Frobenius norm of every group,
 *                         then the k largest (Sec. 4, the Z-subproblem, Eq. 4,
 *                         and its filter-, channel- and shape-wise solutions).
 *   sadmm_pack            Compacts the kept rows (filters) and columns
 *                         ((channel, kt, kh, kw) taps) of the lowered GEMM
 *                         matrix into a dense bf16 matrix plus a gather table
 *                         (Sec. 3, "Combination of structured sparsities":
 *                         filter-wise = row pruning, channel-/shape-wise =
 *                         column pruning; the result is a smaller full matrix).
 *   sadmm_conv_fwd        Implicit GEMM over only the kept rows and columns,
 *                         bias + ReLU fused, written to the full NCHW / NCDHW
 *                         output with every pruned filter's plane set to zero.
 *
 * Conventions for every call:
 *  - All tensor pointers are DEVICE pointers owned by the caller.  The library
 *    never allocates device memory and never synchronises the stream, except
 *    sadmm_last_device_status, which synchronises to read the device flag.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  All work is
 *    enqueued on it, in order, asynchronously.  The kernels are launched with
 *    programmatic stream serialization: one may be scheduled while the kernel
 *    before it on the stream finishes, and it waits for that kernel to complete
 *    before it reads or writes global memory, so stream order is kept.
 *  - Arguments are validated on the host before any launch; a bad argument
 *    returns SADMM_EINVAL and enqueues nothing.  A failed launch returns
 *    SADMM_ECUDA.  Shapes the kernels do not support (see each call) return
 *    SADMM_EUNSUPPORTED.  There is no CPU fallback.
 *  - Layouts are dense row-major (C order): W is [F][Cg][KT][KH][KW]
 *    (OIDHW, KT = 1 for 2-D, Cg = C / groups), x is [N][C][T][H][W], y is
 *    [N][F][OT][OH][OW].  Dilation is 1.
 */
#ifndef SADMM_H
#define SADMM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SADMM_ABI_VERSION 6

/* Most layers one batched call (sadmm_project_groups_batch,
 * sadmm_admm_update_batch) takes. */
#define SADMM_MAX_BATCH 64

/* Bytes of the fixed device array of sadmm_project_groups_noalloc. */
#define SADMM_NOALLOC_SCRATCH_BYTES (256 * 1024)

typedef enum {
    SADMM_OK = 0,
    SADMM_EINVAL = -1,       /* bad argument, shape or buffer size          */
    SADMM_ECUDA = -2,        /* a CUDA runtime call or launch failed        */
    SADMM_ETIMEOUT = -3,     /* a device-side wait ran past its limit       */
    SADMM_EUNSUPPORTED = -4, /* valid request outside what the kernels do   */
    SADMM_EBOUNDS = -5       /* debug build: a device-side index check failed */
} sadmm_status;

typedef enum { SADMM_BF16 = 0, SADMM_FP32 = 1 } sadmm_dtype;

/* Column (GEMM-column) pruning kind.  Filter (row) pruning is always
 * available through k_filters / n_filt and combines with any of these. */
typedef enum {
    SADMM_COL_NONE = 0,    /* keep every column                                  */
    SADMM_COL_SHAPE = 1,   /* shape-wise: groups are single (c,kt,kh,kw) columns */
    SADMM_COL_CHANNEL = 2  /* channel-wise: groups are whole channels c          */
} sadmm_colkind;

/* A CONV layer.  t = kt = st = 1 and pt = 0 for 2-D layers. */
typedef struct {
    int n, c, t, h, w;   /* input: batch, channels, depth, height, width */
    int f, groups;       /* filters (output channels), conv groups       */
    int kt, kh, kw;      /* kernel extent                                */
    int st, sh, sw;      /* strides                                      */
    int pt, ph, pw;      /* zero padding on each side                    */
} sadmm_conv_desc;

/* Execution plan of one pruned layer.  Filled on the host by sadmm_plan_init
 * (sizes) and sadmm_pack (device buffer, TMA descriptor); read-only after.
 * The device buffer `dev` is caller-owned and must stay alive while any
 * sadmm_conv_fwd that uses the plan is in flight.  The struct itself is plain
 * host memory and may be copied. */
typedef struct {
    sadmm_conv_desc desc;
    int n_filt;       /* F': kept filters over all conv groups                */
    int colkind;      /* sadmm_colkind                                        */
    int n_colgroups;  /* kept column groups (columns, or channels)           */
    int n_cols;       /* K': kept GEMM columns (channels x taps if channel)  */
    int k_pad;        /* K' rounded up to a multiple of 64 (at least 64)     */
    int bn;           /* filter rows per tile: multiple of 16, at most 256    */
    int n_tiles;      /* filter tiles per conv group                          */
    int n_pad;        /* rows per conv group in the packed matrix = bn*n_tiles */
    size_t dev_bytes; /* device bytes the plan needs (see sadmm_plan_init)    */
    void* dev;        /* device buffer bound by sadmm_pack                    */
    size_t off_wp, off_gather, off_rowmap, off_zeromap, off_counts, off_colidx;
    size_t off_partial; /* split-K partial sums (when splits > 1)              */
    int splits;         /* K' split over this many CTAs per output tile (>= 1)  */
    int stages_per_split; /* 64-column stages of K' per split                  */
    size_t off_sk;      /* stream-K partial sums and arrival counters (sk_len > 0) */
    int sk_len;         /* stream-K: 64-column stages per CTA (0: whole tiles)  */
    int sk_grid;        /* stream-K: CTAs launched                              */
    int ctas;           /* CTAs a forward launches at most (one per SM)         */
    /* Input-slab forward (xs_mode = 1, see sadmm_plan_init): geometry of the
     * space-to-depth input and of the slab one 128-row tile reads. */
    int xs_mode;        /* 1: the forward runs the slab path                    */
    int xs_r, xs_q;     /* block taps: ceil(KH / sh), ceil(KW / sw)             */
    int xs_cs;          /* slab channels: kept channels * sh * sw, to 16        */
    int xs_hb, xs_wb;   /* block rows / columns: OH + xs_r - 1, OW + xs_q - 1   */
    int xs_pimg;        /* block pixels per image and chunk: xs_hb*xs_wb, to 8  */
    int xs_sp;          /* slab pixels of a tile: 128 + (xs_r-1)*xs_wb + xs_q-1, to 8 */
    int xs_kpad;        /* slab GEMM columns xs_r*xs_q*xs_cs, rounded up to 64  */
    size_t off_xs;      /* space-to-depth input [N][xs_cs/8][xs_pimg][8] bf16   */
    size_t off_wps;     /* slab-ordered packed weights [bn][xs_kpad] bf16       */
    size_t off_scol;    /* slab column -> GEMM column (-1: zero) [xs_kpad] int32,
                           then the kept input channels [xs_cs] int32          */
    uint64_t tmap[16];    /* 128-byte TMA tensor map of the packed matrix       */
    uint64_t tmap_ws[16]; /* TMA map of the slab-ordered weights (xs_mode)      */
    uint64_t tmap_xs[16]; /* TMA map of the space-to-depth input (xs_mode)      */
} sadmm_plan;

/* ------------------------------------------------------------------------ */

/* Library ABI version (SADMM_ABI_VERSION) and sizeof(sadmm_plan), so that
 * bindings can check their mirror of the struct. */
int sadmm_abi_version(void);
size_t sadmm_plan_struct_size(void);

/* Human-readable name of a status code (static string). */
const char* sadmm_status_string(int status);

/* Device bytes of scratch sadmm_project_groups needs for this layer and
 * column kind (keys, counters).  0 on a bad descriptor. */
size_t sadmm_workspace_size(const sadmm_conv_desc* d, int colkind);

/*
 * Euclidean projection onto the structured-sparsity set (Sec. 4, Eq. 4):
 * V = W (+U when U != NULL, the scaled ADMM dual; Sec. 4 projects W + U),
 * squared Frobenius norm O_g of every group, keep the k largest.
 *
 *   W, U       device, dtype `wdt` (bf16 or fp32), layout OIDHW ([F][K] as a
 *              GEMM matrix, K = Cg*KT*KH*KW).  U may be NULL.
 *   k_filters  filters to keep, 0..F (F = no filter pruning).
 *   colkind    SADMM_COL_NONE / SHAPE / CHANNEL.
 *   k_cols     column groups to keep: 0..K (shape) or 0..Cg (channel); ignored
 *              for SADMM_COL_NONE.
 *   filt_idx   device int32 [k_filters]: kept filters, ascending.
 *   col_idx    device int32 [k_cols]: kept columns (shape) or channels
 *              (channel), ascending.  May be NULL for SADMM_COL_NONE.
 *   keys_out   optional device fp64 [F + G]: filter keys, then column-group
 *              keys (G = K or Cg; 0 for SADMM_COL_NONE).
 *   workspace  device scratch of at least sadmm_workspace_size() bytes.
 *
 * Combined row and column pruning: filters are chosen first on the full
 * tensor, then column keys are summed over the kept filters only.  Equal keys
 * go to the lower group index.  Keys are fp64 sums of exact fp64 squares;
 * the order of equal-key groups is resolved by index, so the index lists are
 * deterministic.  Grouped convs: a filter group is one filter among all F; a
 * column group spans all F filters (the same column set serves every conv
 * group).  A kind kept whole (k_filters = F, or k_cols = G) with keys_out
 * NULL skips its keys: its list is 0..F-1 (0..G-1), exactly the top-k.
 */
sadmm_status sadmm_project_groups(const sadmm_conv_desc* d, const void* W, const void* U,
                                  int wdt, int k_filters, int colkind, int k_cols,
                                  int* filt_idx, int* col_idx, double* keys_out,
                                  void* workspace, size_t ws_bytes, void* stream);

/*
 * One layer of a batched projection (sadmm_project_groups_batch): the
 * arguments of sadmm_project_groups for that layer, its own workspace
 * included.
 */
typedef struct {
    sadmm_conv_desc desc;
    const void* W;
    const void* U;         /* may be NULL */
    int k_filters, colkind, k_cols;
    int* filt_idx;
    int* col_idx;
    double* keys_out;      /* may be NULL */
    void* workspace;
    size_t ws_bytes;
} sadmm_project_item;

/*
 * sadmm_project_groups for n layers at once (1 <= n <= SADMM_MAX_BATCH), all
 * of dtype `wdt` (Sec. 4: an ADMM iteration projects every layer).  Results
 * are those of n separate calls, bit for bit; the work of all layers shares
 * each launch (filter keys, the layers' row selects side by side, column
 * keys, the column selects side by side), so a batch costs about what one
 * small layer does.  Each item is checked as sadmm_project_groups checks its
 * arguments; any bad item gives SADMM_EINVAL and nothing is enqueued.  The
 * items' outputs and workspaces must not overlap.
 */
sadmm_status sadmm_project_groups_batch(const sadmm_project_item* items, int n, int wdt, void* stream);

/* Device bytes of scratch sadmm_admm_update needs for this layer and column
 * kind (the projection's keys plus row and column keep flags).  0 on a bad
 * descriptor. */
size_t sadmm_admm_workspace_size(const sadmm_conv_desc* d, int colkind);

/*
 * One ADMM Z- and U-update of a layer (Sec. 4): the Z-subproblem is solved by
 * the Euclidean projection of V = W^{k+1} + U^k onto the structured-sparsity
 * set, then the scaled dual becomes U^{k+1} = U^k + W^{k+1} - Z^{k+1}.
 *
 *   W       device [F][K] (OIDHW), dtype `wdt` (bf16 or fp32): W^{k+1}, read.
 *   U       device [F][K], same dtype: U^k on entry, U^{k+1} on return.
 *   Z       device [F][K], same dtype: Z^{k+1}, every element written.
 *   k_filters, colkind, k_cols, filt_idx, col_idx, keys_out: as in
 *           sadmm_project_groups, on V (the kept lists are returned too).
 *   workspace  device scratch of at least sadmm_admm_workspace_size() bytes,
 *           256-byte aligned.
 *
 * V is formed once in the tensors' precision (fp32 add, or bf16 inputs added
 * in fp32 and rounded to nearest even); group keys use V widened exactly to
 * fp64 as in sadmm_project_groups.  Z = V on every kept (filter, column) pair
 * and 0 elsewhere; U^{k+1} = V - Z: 0 on the kept pairs and V elsewhere.
 * W, U and Z must not overlap (SADMM_EINVAL).  F above 65535 gives
 * SADMM_EUNSUPPORTED.
 */
sadmm_status sadmm_admm_update(const sadmm_conv_desc* d, const void* W, void* U, void* Z, int wdt,
                               int k_filters, int colkind, int k_cols, int* filt_idx, int* col_idx,
                               double* keys_out, void* workspace, size_t ws_bytes, void* stream);

/*
 * One layer of a batched ADMM update (sadmm_admm_update_batch): the
 * arguments of sadmm_admm_update for that layer.
 */
typedef struct {
    sadmm_conv_desc desc;
    const void* W;
    void* U;
    void* Z;
    int k_filters, colkind, k_cols;
    int* filt_idx;
    int* col_idx;
    double* keys_out;      /* may be NULL */
    void* workspace;       /* sadmm_admm_workspace_size() bytes, 256-byte aligned */
    size_t ws_bytes;
} sadmm_admm_item;

/*
 * sadmm_admm_update for n layers at once (1 <= n <= SADMM_MAX_BATCH), all of
 * dtype `wdt`: one ADMM Z- and U-update of every layer of a network (Sec. 4).
 * Results equal those of n separate calls bit for bit; the batch shares the
 * projection's launches (see sadmm_project_groups_batch) and one apply pass.
 * Each item is checked as sadmm_admm_update checks its arguments (SADMM_EINVAL
 * before anything is enqueued).  Tensors of different items must not overlap.
 */
sadmm_status sadmm_admm_update_batch(const sadmm_admm_item* items, int n, int wdt, void* stream);

/* Device bytes of scratch the non-structured projection needs for this
 * layer (selection state, a 2048-bin histogram, one counter per 4096
 * weights).  0 on a bad descriptor. */
size_t sadmm_elements_workspace_size(const sadmm_conv_desc* d);

/*
 * Non-structured projection (Sec. 4, non-structured weight sparsity): keep the
 * k_elems entries of V = W (+U) with the largest magnitudes |V|, zero the rest.
 * |V| is compared exactly (V formed in fp64); equal magnitudes go to the lower
 * flat index a*K + j (the reading used for every top-k in this library).
 *
 *   W, U      device [F][K], dtype `wdt`; U may be NULL.
 *   k_elems   0 .. F*K.
 *   keep_out  device uint8 [F*K]: 1 for a kept entry, 0 otherwise.
 *   workspace sadmm_elements_workspace_size() bytes, 256-byte aligned.
 * The paper finds this sparsity hard to speed up on a GPU (Sec. 5, cuSPARSE);
 * sadmm_sparse_conv_fwd below runs such a layer, for that comparison.
 */
sadmm_status sadmm_project_elements(const sadmm_conv_desc* d, const void* W, const void* U, int wdt,
                                    long long k_elems, unsigned char* keep_out, void* workspace,
                                    size_t ws_bytes, void* stream);

/*
 * The ADMM Z- and U-update for non-structured sparsity (Sec. 4): Z = the
 * k_elems largest-magnitude entries of V = W + U (V rounded once to the
 * tensors' precision, as in sadmm_admm_update), U <- V - Z.  W, U, Z as in
 * sadmm_admm_update (no overlap); workspace as for sadmm_project_elements.
 */
sadmm_status sadmm_admm_update_elements(const sadmm_conv_desc* d, const void* W, void* U, void* Z, int wdt,
                                        long long k_elems, void* workspace, size_t ws_bytes, void* stream);

/*
 * Forward of a layer pruned element by element (non-structured sparsity, Sec. 4;
 * the comparison of the paper's speed tests, Sec. 5, where such layers run
 * through a sparse library and gain little or lose on a GPU).  The kept
 * weights are stored per filter in compressed rows (CSR) and the forward runs
 * on the CUDA cores, one thread per output pixel and filter: a sparse matrix
 * has no dense tile for the tensor cores.  It exists to measure that contrast
 * on this GPU beside sadmm_conv_fwd at the same density.
 *
 * sadmm_sparse_plan_size: device bytes of a plan holding up to `capacity` kept
 *   weights (0 .. F*K): row pointers [F + 1] int32 (rounded up to 256 B), then
 *   `capacity` 16-byte entries {x offset of the column, tap bits, fp32 weight}.
 *   0 on a bad descriptor or capacity.
 * sadmm_sparse_pack: builds the plan from W (bf16 or fp32, OIDHW) and a keep
 *   mask (device uint8 [F][K], nonzero = kept; e.g. from
 *   sadmm_project_elements).  plan: device, 256-byte aligned, at least
 *   sadmm_sparse_plan_size bytes.  More kept weights than `capacity` give an
 *   empty plan (its forward writes ReLU(bias)) and raise the device status
 *   word (SADMM_EINVAL from sadmm_last_device_status).  F above 65535 gives
 *   SADMM_EUNSUPPORTED.
 * sadmm_sparse_conv_fwd: y[n, f, o] = ReLU(bias[f] + sum over the kept (f, col)
 *   of W[f][col] * x at col's tap, zero outside the input), fp32 accumulation
 *   in column order; x, bias, relu, y and ydt as in sadmm_conv_fwd.  No filter
 *   is pruned as a whole here, so the bias is never masked.
 */
size_t sadmm_sparse_plan_size(const sadmm_conv_desc* d, long long capacity);
sadmm_status sadmm_sparse_pack(const sadmm_conv_desc* d, const void* W, int wdt, const unsigned char* keep,
                               long long capacity, void* plan, size_t plan_bytes, void* stream);
sadmm_status sadmm_sparse_conv_fwd(const sadmm_conv_desc* d, const void* plan, const void* x, const float* bias,
                                   int relu, void* y, int ydt, void* stream);

/*
 * Sizes a plan for `n_filt` kept filters and `n_colgroups` kept column groups
 * (columns or channels) of kind `colkind`.  Fills every size field of `plan`,
 * including plan->dev_bytes, the device buffer sadmm_pack needs.  Host only;
 * enqueues nothing.  SADMM_EUNSUPPORTED when the packed row count per conv
 * group would exceed 4096 or K' would exceed 8192.
 *
 * Small batches (the paper times batch 1, Sec. 5): when the layer has fewer
 * output tiles (128 pixels x one filter tile of one conv group) than the
 * current device has SMs, K' is split over plan->splits CTAs per tile (at
 * least two 64-column stages per split when K' has at most eight); each
 * writes fp32 partial sums to a region of the plan's device buffer and a
 * second kernel adds them in split order, then applies bias and ReLU.  The
 * split depends on the current device's SM count and is fixed in the plan.
 *
 * Tail balance (stream-K): when the output tiles do not divide evenly over the
 * SMs and an even share of the tiles' 64-column stages (plan->sk_len per CTA,
 * plan->sk_grid CTAs) shortens the busiest CTA's work by at least 1/8, each
 * CTA takes a contiguous run of stages instead of whole tiles (only when a
 * tile's accumulator fits TMEM twice and K' is at least 4 * bn, where the cost
 * of a cut tile measured below its gain).  A tile cut at
 * a run boundary is finished by whichever of its two CTAs arrives last: both
 * write fp32 partial sums to the plan's buffer, an arrival counter there
 * (reset by the last arrival; zeroed by sadmm_pack) tells the second which
 * it is, and it adds the two halves in K' order, then bias and ReLU.  After a
 * device-side failure (sadmm_last_device_status) the plan must be packed again.
 */
/*
 * Input-slab path (plan->xs_mode = 1): a 2-D layer with one conv group, at
 * most 256 kept filters and every column of its kept channels kept (no
 * column pruning, or whole channels pruned), whose kept channels times
 * sh * sw come to at most 64, with more than one block tap (xs_r * xs_q >= 2)
 * and a slab GEMM at most twice as wide as K' -- the first layer of a
 * network, typically (the paper keeps AlexNet's
 * CONV1 whole).  The forward then first rewrites x as a space-to-depth copy
 * in the plan's buffer: block pixel (hb, wb) holds, for each kept channel c
 * and phase (a, b) < (sh, sw), the input x[c][hb*sh + a - ph][wb*sw + b - pw]
 * (zero outside), which turns the strided KH x KW conv into a stride-1
 * xs_r x xs_q conv over xs_cs channels.  A tile of 128 consecutive block
 * pixels of one image (output rows of xs_wb pixels, the last xs_q - 1 of
 * each discarded) reads one contiguous slab of block pixels, loaded once into
 * shared memory; each block tap (r, q) is the slab shifted by r * xs_wb + q
 * pixels, fed to the tensor cores directly (the pixels on the MMA's M side,
 * the kept filters on its N side), so no im2col copy is built.  The
 * slab GEMM has xs_r * xs_q * xs_cs columns (the taps and channels past the
 * kernel or the kept channels hold zero weights): the same sums as the
 * gathered path, in another order.  No K' split or stream-K in this path.
 */
sadmm_status sadmm_plan_init(sadmm_plan* plan, const sadmm_conv_desc* d,
                             int n_filt, int colkind, int n_colgroups);

/*
 * sadmm_plan_init for a forward that may occupy at most `max_ctas` SMs
 * (0 or above the SM count: all of them).  The conv kernel keeps one CTA per
 * SM for its whole run, so nothing else runs beside it; a cap leaves
 * SM count - max_ctas SMs to work on other streams (the next layers'
 * projection and pack, say).  The split-K and stream-K choices, and so the
 * plan's device bytes, follow the cap.  Results do not depend on it.
 */
sadmm_status sadmm_plan_init_ctas(sadmm_plan* plan, const sadmm_conv_desc* d,
                                  int n_filt, int colkind, int n_colgroups, int max_ctas);

/*
 * Compacts the kept weights (Sec. 3, row/column pruning of the GEMM matrix):
 *   Wp[g][i][j] = bf16(W[f_i][col_j]) for the i-th kept filter f_i of conv
 *   group g and the j-th kept column, zero beyond the kept counts;
 *   a gather table entry per kept column (its channel offset in x and its
 *   (kt,kh,kw) tap); per conv group the list of kept and of pruned filters.
 *
 *   filt_idx  device int32 [plan->n_filt], ascending, in [0,F); NULL when
 *             n_filt == F (all filters).
 *   col_idx   device int32 [plan->n_colgroups], ascending: columns in [0,K)
 *             (shape) or channels in [0,Cg) (channel); NULL for COL_NONE.
 *   dev       device buffer of >= plan->dev_bytes bytes, 256-byte aligned;
 *             becomes plan->dev.
 * Writes the TMA descriptor of Wp into plan->tmap.  For a slab plan it also
 * packs the weights in slab column order (plan->off_wps, plan->tmap_ws) and
 * writes the TMA map of the space-to-depth input (plan->tmap_xs).  Index lists
 * are checked on the device: a list that is not strictly ascending or holds an
 * index out of range gives a plan with every filter pruned and every column
 * dropped (its forward writes an all-zero output) and raises the device status
 * word, which the next sadmm_last_device_status returns as SADMM_EINVAL.
 */
sadmm_status sadmm_pack(sadmm_plan* plan, const void* W, int wdt,
                        const int* filt_idx, const int* col_idx,
                        void* dev, size_t dev_bytes, void* stream);

/*
 * sadmm_pack for a batch of layers (1 .. SADMM_MAX_BATCH items, one plan each,
 * every W of type wdt): the same plans, buffers, descriptors and device checks
 * as n sadmm_pack calls, with two kernel launches for the whole batch (the
 * meta data of every layer, then the packed rows of every layer).  Each item's
 * fields are as the arguments of sadmm_pack; a bad item returns SADMM_EINVAL
 * and enqueues nothing.
 */
typedef struct {
    sadmm_plan* plan;
    const void* W;
    const int* filt_idx;
    const int* col_idx;
    void* dev;
    size_t dev_bytes;
} sadmm_pack_item;
sadmm_status sadmm_pack_batch(sadmm_pack_item* items, int n, int wdt, void* stream);

/*
 * Pruned CONV forward (Sec. 3: the pruned layer is a smaller full GEMM):
 *   y[n, f, o] = ReLU(bias[f] + sum_{j < K'} Wp[f][j] * x[n, g*Cg + c_j,
 *                ot*st-pt+kt_j, oh*sh-ph+kh_j, ow*sw-pw+kw_j])   f kept,
 *   y[n, f, o] = 0                                                f pruned,
 * x outside the input reads as zero.  bf16 x bf16 products accumulate in fp32
 * (tcgen05 MMA, TMEM accumulator).
 *
 *   x     device bf16 [N][C][T][H][W]; element (2-byte) aligned (SADMM_EINVAL
 *         otherwise): the kernels read x one element at a time.
 *   bias  device fp32 [F] or NULL (zero).
 *   relu  nonzero: apply ReLU.
 *   y     device [N][F][OT][OH][OW] of dtype `ydt` (fp32 or bf16, rounded
 *         to nearest even); every element is written.
 * Requires sm_100-family tensor cores (SADMM_EUNSUPPORTED otherwise) and
 * N*C*T*H*W < 2^31.  Launches that use one plan must not overlap on the GPU
 * (stream-ordered is fine): split-K partial sums, stream-K arrival
 * counters and the slab path's space-to-depth input live in the plan's
 * buffer.
 */
sadmm_status sadmm_conv_fwd(const sadmm_plan* plan, const void* x, const float* bias,
                            int relu, void* y, int ydt, void* stream);

/*
 * sadmm_conv_fwd in two calls, so that a caller can overlap an input-slab
 * plan's space-to-depth pass with other work (the layer's projection and
 * pack, for the first layer of a network, whose input is ready before its
 * weights are):
 *   SADMM_FWD_INPUT  the space-to-depth pass alone (x read, the plan's copy
 *                    written; nothing for a gathered plan).  Without channel
 *                    pruning it reads nothing sadmm_pack writes, so it may
 *                    run while the plan is being packed again (the plan must
 *                    have been packed once: its buffer is bound); with channel
 *                    pruning it reads the kept-channel list and must follow
 *                    sadmm_pack.
 *   SADMM_FWD_REST   the rest: for a slab plan the conv kernel on the copy
 *                    the last INPUT call wrote (x unused, may be NULL); a
 *                    gathered plan runs whole.
 *   SADMM_FWD_ALL    both (= sadmm_conv_fwd).
 * The caller orders INPUT before REST (same stream, or an event).  Results
 * equal those of sadmm_conv_fwd bit for bit.
 */
typedef enum { SADMM_FWD_ALL = 0, SADMM_FWD_INPUT = 1, SADMM_FWD_REST = 2 } sadmm_fwd_phase;
sadmm_status sadmm_conv_fwd_phase(const sadmm_plan* plan, const void* x, const float* bias,
                                  int relu, void* y, int ydt, int phase, void* stream);

/*
 * sadmm_project_groups without a caller-provided workspace.  The paper has no
 * counterpart: this exists for callers that cannot hand the library device
 * scratch memory -- a plugin or host framework that passes only its input and
 * output tensors and keeps every allocation to itself, or a serving loop that
 * must not allocate (nor risk running out of memory) once it is running.
 *
 * Arguments and results are those of sadmm_project_groups without
 * `workspace` / `ws_bytes`.  The group keys go to one fixed device array
 * compiled into the library, SADMM_NOALLOC_SCRATCH_BYTES (256 KiB) on every
 * GPU that loads the library, held until the process exits.  A layer
 * whose keys need more (sadmm_workspace_size() above that) is rejected with
 * SADMM_EUNSUPPORTED before anything is enqueued.  Exactly: a layer fits when
 * round_up(F, 32) + round_up(K, 32) <= 16352, K = Cg*KT*KH*KW, whatever the
 * column kind (e.g. F = 192 filters with K = 16160 columns, or F = 16320 with
 * K = 32).  The call allocates nothing: no cudaMalloc, no cudaFree.
 *
 * The first call on a device looks up the array's device address (a host-side
 * CUDA runtime query, once per device, with that device current); make that
 * first call before any stream capture.  The address is kept for the life of
 * the process: after cudaDeviceReset the array is gone and the kept address is
 * stale, so do not call this entry point on a device that has been reset.  Every call shares the array.  Nothing
 * in it needs to start at zero (each key is written before it is read), but
 * calls that overlap on the GPU -- on different streams with no ordering
 * between them -- race on it and can return wrong index lists.
 */
sadmm_status sadmm_project_groups_noalloc(const sadmm_conv_desc* d, const void* W, const void* U,
                                          int wdt, int k_filters, int colkind, int k_cols,
                                          int* filt_idx, int* col_idx, double* keys_out,
                                          void* stream);

/* Device bytes of scratch for sadmm_conv_bwd to take the layer's output
 * pixels in chunks of at most 32768 (sized so a chunk's gathered bf16
 * operands and fp32 products stay in L2): the default.  0 on a bad plan. */
size_t sadmm_conv_bwd_workspace_size(const sadmm_plan* plan);

/* Device bytes of scratch for chunks of `chunk_pixels` output pixels (rounded
 * up to a multiple of 256, at least 256, at most 32768).  sadmm_conv_bwd
 * accepts any workspace at least the size for 256 pixels and takes the pixels
 * in the largest chunks (up to 32768) the workspace holds: a smaller workspace
 * costs more launches and partial-sum passes, not results (the dW and db
 * reductions keep a fixed order for a given chunk size). */
size_t sadmm_conv_bwd_workspace_size_chunk(const sadmm_plan* plan, long long chunk_pixels);

/*
 * Backward of the packed pruned layer for masked retraining (Sec. 4, "Masked
 * mapping and retraining": the pruned weights stay zero and only the kept ones
 * are trained).  With dZ = dY * [y > 0] when relu is set (else dZ = dY):
 *   dW[f][col] = sum over images and output pixels of dZ * x at (f, col), for
 *                every kept filter f and kept GEMM column col; 0 elsewhere;
 *   db[f]      = sum of dZ over images and pixels for kept f; 0 for pruned f;
 *   dx         = the input gradient through the kept weights only.
 * The contractions run on the tensor cores (bf16 operands, fp32 accumulation);
 * dW and db are summed in a fixed order (deterministic); dx is summed with
 * fp32 atomics (its last bits depend on timing).  For an input-slab plan
 * (plan->xs_mode) with at most 128 kept filters, dW is contracted on the
 * plan's space-to-depth copy of x (rewritten by this call) instead of an
 * im2col copy; its workspace then also holds dZ in the output's block-pixel
 * grid and one fp32 partial dW per CTA.
 *
 *   plan   a packed plan (sadmm_pack) of the layer.
 *   x      device bf16 [N][C][T][H][W] (needed for dW).
 *   dy     device bf16 [N][F][OT][OH][OW].
 *   y      device forward output of dtype ydt (bf16/fp32), read when relu != 0.
 *   dW     device fp32 [F][K] (OIDHW) or NULL; db fp32 [F] or NULL;
 *          dx fp32 [N][C][T][H][W] or NULL.  Every element of each is written.
 *   workspace  ws_bytes of device scratch, 1024-byte aligned: at least
 *          sadmm_conv_bwd_workspace_size_chunk(plan, 256) (else SADMM_EINVAL);
 *          sadmm_conv_bwd_workspace_size(plan) gives the largest chunks.
 */
sadmm_status sadmm_conv_bwd(const sadmm_plan* plan, const void* x, const void* dy, const void* y, int ydt,
                            int relu, float* dW, float* db, float* dx, void* workspace, size_t ws_bytes,
                            void* stream);

/*
 * The tensor-core GEMM the backward uses, for direct use and testing:
 * C[M][N] = (accumulate ? C : 0) + A[M][K] * B[N][K]^T with bf16 A and B
 * (row-major, K contiguous), fp32 C (row stride ldc).  M % 128 == 0,
 * K % 64 == 0, N a multiple of 16, ldc % 4 == 0, 16-byte aligned pointers.
 */
sadmm_status sadmm_gemm_bf16(const void* A, const void* B, float* C, long long M, long long N, long long K,
                             long long ldc, int accumulate, void* stream);

/*
 * Failure-detection self-test; the paper has no counterpart.  Runs, in one
 * CTA on `stream`, the bounded mbarrier wait every pipelined kernel here uses,
 * with a limit of `limit_us` microseconds (1 .. 1000000) instead of the
 * kernels' 4 s.  With `arrive` = 0 nothing ever arrives on the barrier: the
 * wait gives up after the limit, raises the device status word (so the next
 * sadmm_last_device_status returns SADMM_ETIMEOUT) and the kernel returns,
 * leaving the context usable.  With `arrive` != 0 the barrier completes first
 * and the wait succeeds.  `result` (device int, optional): 1 when the wait saw
 * its phase complete, 0 when it gave up.  Nothing here faults or hangs.
 */
sadmm_status sadmm_selftest_wait(unsigned int limit_us, int arrive, int* result, void* stream);

/*
 * Synchronises `stream`, then reports and clears the device status word that
 * the kernels set when a bounded wait expires (SADMM_ETIMEOUT), a device-side
 * check of an index list fails (SADMM_EINVAL) or, in a library built with
 * -DSADMM_DEBUG, an index check of a global load or store fails
 * (SADMM_EBOUNDS: the access was skipped, a load read zero).  SADMM_OK when
 * clear.
 */
sadmm_status sadmm_last_device_status(void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SADMM_H */
