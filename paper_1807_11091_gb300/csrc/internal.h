// internal.h -- host-side declarations shared by the libsadmm translation units.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "sadmm.h"

namespace sadmm {

// Derived sizes of a validated descriptor.
struct Geometry {
    long long n, c, t, h, w, f, groups, kt, kh, kw, st, sh, sw, pt, ph, pw;
    long long cg, fg, taps, k;      // K = Cg * taps GEMM columns
    long long ot, oh, ow, plane, m; // output extents, pixels per image, N * plane
};

// Checks a descriptor; fills `g` on success.
sadmm_status check_desc(const sadmm_conv_desc* d, Geometry* g);

// The argument checks every projection entry point shares (sadmm_project_groups,
// its no-workspace variant, sadmm_admm_update): W and filt_idx present, a known
// dtype and column kind, k_filters in [0, F], k_cols in [0, G] with col_idx
// present when columns are pruned, keys_out 8-byte aligned.  Each entry point
// then checks its own workspace.
sadmm_status check_project_args(const Geometry& g, const void* W, int wdt, int k_filters, int colkind, int k_cols,
                                const int* filt_idx, const int* col_idx, const double* keys_out);

// A named NVTX range around one entry point (seen by nsys / ncu range filters;
// costs one branch when no tool is attached).
struct NvtxRange {
    explicit NvtxRange(const char* name);
    ~NvtxRange();
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};

// Address of the device status word on the current device (cached per device).
int* device_status_ptr();

// Number of SMs of the current device (cached per device).
int device_sm_count();

// Compute capability major of the current device (cached per device).
int device_cc_major();

// Rounds x up to a multiple of a.
inline long long round_up(long long x, long long a) { return (x + a - 1) / a * a; }

// ---- projection (project.cu) ----
size_t project_workspace_bytes(const Geometry& g, int colkind);

// One layer of a batched projection or ADMM update: its geometry, tensors,
// selection, index lists and workspace; rkeep / ckeep (optional) get a byte
// per filter / column group; Z is the ADMM update's output (NULL otherwise).
struct ProjItem {
    Geometry g;
    const void* W;
    const void* U;
    void* Z;
    int k_filters, colkind, k_cols;
    int* filt_idx;
    int* col_idx;
    double* keys_out;
    void* ws;
    uint8_t* rkeep;
    uint8_t* ckeep;
};
constexpr int kMaxBatch = SADMM_MAX_BATCH;
// The projection of items[0..n) (checked arguments, one dtype): one launch per
// phase for the whole batch.
sadmm_status launch_project_batch(const ProjItem* items, int n, int wdt, cudaStream_t s);
// The ADMM update of items[0..n): the batched projection with keep flags in
// each item's workspace, then one apply pass over every layer.
sadmm_status launch_admm_batch(const ProjItem* items, int n, int wdt, cudaStream_t s);
// rkeep / ckeep (optional): a byte per filter / per column group, 1 when kept.
sadmm_status launch_project(const Geometry& g, const void* W, const void* U, int wdt, int k_filters,
                            int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out,
                            void* ws, cudaStream_t s, uint8_t* rkeep = nullptr, uint8_t* ckeep = nullptr);

// ---- ADMM Z/U update (admm.cu) ----
size_t admm_workspace_bytes(const Geometry& g, int colkind);
sadmm_status launch_admm_update(const Geometry& g, const void* W, void* U, void* Z, int wdt, int k_filters,
                                int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out, void* ws,
                                cudaStream_t s);

// ---- non-structured projection (elements.cu) ----
size_t elements_workspace_bytes(const Geometry& g);
// keep_out (optional) and/or the ADMM update (Z and U non-null).
sadmm_status launch_elements(const Geometry& g, const void* W, void* U, void* Z, int wdt, long long k,
                             uint8_t* keep_out, void* ws, cudaStream_t s);

// ---- non-structured sparse forward (sparse.cu) ----
// Plan buffer: row pointers [F + 1] int32 (to 256 B), then `capacity` entries of 16 B.
size_t sparse_plan_bytes(const Geometry& g, long long capacity);
sadmm_status launch_sparse_pack(const Geometry& g, const void* W, int wdt, const uint8_t* keep, void* buf,
                                long long capacity, cudaStream_t s);
sadmm_status launch_sparse_conv(const Geometry& g, const void* buf, const void* x, const float* bias, int relu,
                                void* y, int ydt, cudaStream_t s);

// ---- generic bf16 GEMM on the tensor cores (gemm.cu) ----
// C[M][N] (fp32, row stride ldc floats) = (accumulate ? C : 0) + A[M][K] * B[N][K]^T,
// A and B bf16 row-major (K contiguous, row stride K).  M % 128 == 0,
// N % bn == 0, bn a multiple of 16 in [16, 256], K % 64 == 0, ldc % 4 == 0,
// A, B and C 16-byte aligned.
// splits > 1: K is cut into `splits` equal ranges (K/64 divisible by splits),
// one CTA per (tile, range).  slice == 0: each adds its product into C with
// fp32 atomics (C must hold the starting value; `accumulate` is then implied).
// slice > 0 (at least M * ldc): range z writes (accumulate: adds) its product
// into its own slice C + z * slice, without atomics; the caller sums them.
sadmm_status launch_gemm(const void* A, const void* B, float* C, long long M, long long N, long long K,
                         long long ldc, int bn, bool accumulate, cudaStream_t s, int splits = 1,
                         long long slice = 0);

// ---- masked-retraining backward (bwd.cu) ----
// Workspace of chunks of `chunk` output pixels (0: the default, the whole
// layer up to 32768 pixels); the smallest chunk is 256 pixels.
size_t bwd_workspace_bytes(const sadmm_plan* plan, const Geometry& g, long long chunk = 0);
sadmm_status launch_conv_bwd(const sadmm_plan* plan, const Geometry& g, const void* x, const void* dy, const void* y,
                             int ydt, int relu, float* dW, float* db, float* dx, void* ws, size_t ws_bytes,
                             cudaStream_t s);

// ---- weight gradient of an input-slab plan (bwd_slab.cu) ----
// Whether the plan's weight gradient runs on the slab (one conv group, at most
// 128 kept filters, at most 512 slab columns); the workspace it needs (0 when
// it does not apply); and the run: the space-to-depth pass of x into the
// plan's copy, dZ in the output's block-pixel grid, the GEMM into per-CTA
// slices and their ordered sum into dW (which the caller has zeroed).
bool wgrad_slab_ok(const sadmm_plan* plan, const Geometry& g);
size_t wgrad_slab_bytes(const sadmm_plan* plan, const Geometry& g);
sadmm_status launch_wgrad_slab(const sadmm_plan* plan, const Geometry& g, const void* x, const void* dy,
                               const void* y, int ydt, int relu, float* dW, void* ws, cudaStream_t s);

// ---- pack (pack.cu) ----
// One layer of a pack launch: its plan (dev bound), geometry, weights and
// index lists (validated on the host as for sadmm_pack).
struct PackJob {
    sadmm_plan* plan;
    Geometry g;
    const void* W;
    const int* filt_idx;
    const int* col_idx;
};
// Packs n layers (1 .. kMaxBatch) with two kernel launches, then encodes each
// plan's TMA descriptors on the host.
sadmm_status launch_pack_batch(const PackJob* jobs, int n, int wdt, cudaStream_t s);

// TMA descriptors of a slab plan's weights and space-to-depth input (host only).
sadmm_status launch_pack_slab(sadmm_plan* plan, const Geometry& g);

// ---- input-slab forward (conv_slab.cu) ----
// Shared-memory stages (one tile's slab each) the slab kernel can hold with
// the weights resident; below 2 the slab path is not available.
int slab_stages(int bn, int kpad_s, int cs, int sp);
// phase: SADMM_FWD_ALL, SADMM_FWD_INPUT (the space-to-depth pass) or
// SADMM_FWD_REST (the conv kernel on the copy the last input pass wrote).
sadmm_status launch_conv_slab(const sadmm_plan* plan, const Geometry& g, const void* x, const float* bias, int relu,
                              void* y, int ydt, int phase, cudaStream_t s);

// ---- forward (conv_fwd.cu) ----
sadmm_status launch_conv_fwd(const sadmm_plan* plan, const Geometry& g, const void* x, const float* bias,
                             int relu, void* y, int ydt, int phase, cudaStream_t s);

// Tap-mask encoding of the gather table: 0 = one bit per tap (at most 31
// taps), 1 = (kt,kh) row bits 0..15 and kw bits 16..30.  Bit 31 marks padding
// columns and is never valid.
inline int tap_mask_mode(const Geometry& g) { return g.taps <= 31 ? 0 : 1; }

}  // namespace sadmm
