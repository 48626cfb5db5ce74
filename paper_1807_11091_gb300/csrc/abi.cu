// abi.cu -- the extern "C" entry points of libsadmm: host-side validation,
// plan sizing and the device status word.  Every entry point checks its
// arguments before enqueuing anything and never synchronises, except
// sadmm_last_device_status.
#include <nvtx3/nvToolsExt.h>
#include <string.h>

#include "common.cuh"
#include "internal.h"

namespace sadmm {

__device__ int g_status_word;

namespace {
constexpr int kMaxDevices = 64;
int* g_status_ptr[kMaxDevices];
int g_sm_count[kMaxDevices];
int g_cc_major[kMaxDevices];

int current_device()
{
    int d = 0;
    if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return 0;
    return d;
}
}  // namespace

int* device_status_ptr()
{
    const int d = current_device();
    if (!g_status_ptr[d]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) == cudaSuccess) g_status_ptr[d] = static_cast<int*>(p);
    }
    return g_status_ptr[d];
}

int device_sm_count()
{
    const int d = current_device();
    if (!g_sm_count[d]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, d);
        g_sm_count[d] = v > 0 ? v : 1;
    }
    return g_sm_count[d];
}

int device_cc_major()
{
    const int d = current_device();
    if (!g_cc_major[d]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrComputeCapabilityMajor, d);
        g_cc_major[d] = v;
    }
    return g_cc_major[d];
}

sadmm_status check_desc(const sadmm_conv_desc* d, Geometry* g)
{
    if (!d || !g) return SADMM_EINVAL;
    const long long v[16] = {d->n,  d->c,  d->t,  d->h,  d->w,  d->f,  d->groups, d->kt,
                             d->kh, d->kw, d->st, d->sh, d->sw, d->pt, d->ph,     d->pw};
    for (int i = 0; i < 13; ++i)
        if (v[i] < 1) return SADMM_EINVAL;
    for (int i = 13; i < 16; ++i)
        if (v[i] < 0) return SADMM_EINVAL;
    Geometry r;
    r.n = d->n; r.c = d->c; r.t = d->t; r.h = d->h; r.w = d->w; r.f = d->f; r.groups = d->groups;
    r.kt = d->kt; r.kh = d->kh; r.kw = d->kw; r.st = d->st; r.sh = d->sh; r.sw = d->sw;
    r.pt = d->pt; r.ph = d->ph; r.pw = d->pw;
    if (r.c % r.groups != 0 || r.f % r.groups != 0) return SADMM_EINVAL;
    r.cg = r.c / r.groups;
    r.fg = r.f / r.groups;
    r.taps = r.kt * r.kh * r.kw;
    r.k = r.cg * r.taps;
    if (r.t + 2 * r.pt < r.kt || r.h + 2 * r.ph < r.kh || r.w + 2 * r.pw < r.kw) return SADMM_EINVAL;
    r.ot = (r.t + 2 * r.pt - r.kt) / r.st + 1;
    r.oh = (r.h + 2 * r.ph - r.kh) / r.sh + 1;
    r.ow = (r.w + 2 * r.pw - r.kw) / r.sw + 1;
    r.plane = r.ot * r.oh * r.ow;
    r.m = r.n * r.plane;
    // index arithmetic limits of the kernels (32-bit offsets inside a tensor)
    if (r.n * r.c * r.t * r.h * r.w >= (1ll << 31)) return SADMM_EUNSUPPORTED;
    if (r.f * r.k >= (1ll << 31) || r.f * r.plane >= (1ll << 31) || r.m >= (1ll << 40)) return SADMM_EUNSUPPORTED;
    // tap-validity masks: one bit per tap, or 16 row bits + 15 kw bits
    if (r.taps > 31 && (r.kt * r.kh > 16 || r.kw > 15)) return SADMM_EUNSUPPORTED;
    if (r.groups > 64) return SADMM_EUNSUPPORTED;
    *g = r;
    return SADMM_OK;
}

sadmm_status check_project_args(const Geometry& g, const void* W, int wdt, int k_filters, int colkind, int k_cols,
                                const int* filt_idx, const int* col_idx, const double* keys_out)
{
    if (!W || !filt_idx) return SADMM_EINVAL;
    if (wdt != SADMM_BF16 && wdt != SADMM_FP32) return SADMM_EINVAL;
    if (colkind != SADMM_COL_NONE && colkind != SADMM_COL_SHAPE && colkind != SADMM_COL_CHANNEL)
        return SADMM_EINVAL;
    if (k_filters < 0 || k_filters > g.f) return SADMM_EINVAL;
    if (colkind != SADMM_COL_NONE) {
        const long long G = (colkind == SADMM_COL_SHAPE) ? g.k : g.cg;
        if (k_cols < 0 || k_cols > G || !col_idx) return SADMM_EINVAL;
    }
    if (keys_out && (reinterpret_cast<uintptr_t>(keys_out) & 7) != 0) return SADMM_EINVAL;
    return SADMM_OK;
}

NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

namespace {
// One CTA runs the kernels' bounded mbarrier wait (mbar_wait_for) on a barrier
// of one expected arrival.  With `arrive` set, thread 0 arrives first and the
// wait must succeed at once; otherwise nothing ever arrives and the wait must
// give up after limit_ns, raise the status word and return.  The result of the
// wait (1 completed, 0 gave up) goes to `out` when it is not NULL.
__global__ void k_selftest_wait(int* status, unsigned long long limit_ns, int arrive, int* out)
{
    __shared__ uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (arrive) mbar_arrive(&bar);
        const bool ok = mbar_wait_for(&bar, 0, &abort_flag, status, limit_ns);
        if (out) *out = ok ? 1 : 0;
    }
}
}  // namespace

}  // namespace sadmm

using namespace sadmm;

extern "C" {

int sadmm_abi_version(void) { return SADMM_ABI_VERSION; }

size_t sadmm_plan_struct_size(void) { return sizeof(sadmm_plan); }

const char* sadmm_status_string(int status)
{
    switch (status) {
    case SADMM_OK: return "ok";
    case SADMM_EINVAL: return "invalid argument";
    case SADMM_ECUDA: return "CUDA error";
    case SADMM_ETIMEOUT: return "device wait timed out";
    case SADMM_EUNSUPPORTED: return "unsupported";
    default: return "unknown status";
    }
}

size_t sadmm_workspace_size(const sadmm_conv_desc* d, int colkind)
{
    Geometry g;
    if (check_desc(d, &g) != SADMM_OK) return 0;
    return project_workspace_bytes(g, colkind);
}

sadmm_status sadmm_project_groups(const sadmm_conv_desc* d, const void* W, const void* U, int wdt,
                                  int k_filters, int colkind, int k_cols, int* filt_idx, int* col_idx,
                                  double* keys_out, void* workspace, size_t ws_bytes, void* stream)
{
    NvtxRange range("sadmm_project_groups");
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    st = check_project_args(g, W, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out);
    if (st != SADMM_OK) return st;
    if (!workspace) return SADMM_EINVAL;
    if (ws_bytes < project_workspace_bytes(g, colkind)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 7) != 0) return SADMM_EINVAL;
    return launch_project(g, W, U, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out, workspace,
                          static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_project_groups_batch(const sadmm_project_item* items, int n, int wdt, void* stream)
{
    NvtxRange range("sadmm_project_groups_batch");
    if (!items || n < 1 || n > SADMM_MAX_BATCH) return SADMM_EINVAL;
    ProjItem pit[SADMM_MAX_BATCH];
    for (int l = 0; l < n; ++l) {
        const sadmm_project_item& it = items[l];
        Geometry g;
        sadmm_status st = check_desc(&it.desc, &g);
        if (st != SADMM_OK) return st;
        st = check_project_args(g, it.W, wdt, it.k_filters, it.colkind, it.k_cols, it.filt_idx, it.col_idx,
                                it.keys_out);
        if (st != SADMM_OK) return st;
        if (!it.workspace || it.ws_bytes < project_workspace_bytes(g, it.colkind)) return SADMM_EINVAL;
        if ((reinterpret_cast<uintptr_t>(it.workspace) & 7) != 0) return SADMM_EINVAL;
        pit[l].g = g;
        pit[l].W = it.W;
        pit[l].U = it.U;
        pit[l].Z = nullptr;
        pit[l].k_filters = it.k_filters;
        pit[l].colkind = it.colkind;
        pit[l].k_cols = it.k_cols;
        pit[l].filt_idx = it.filt_idx;
        pit[l].col_idx = it.col_idx;
        pit[l].keys_out = it.keys_out;
        pit[l].ws = it.workspace;
        pit[l].rkeep = nullptr;
        pit[l].ckeep = nullptr;
    }
    return launch_project_batch(pit, n, wdt, static_cast<cudaStream_t>(stream));
}

size_t sadmm_admm_workspace_size(const sadmm_conv_desc* d, int colkind)
{
    Geometry g;
    if (check_desc(d, &g) != SADMM_OK) return 0;
    return admm_workspace_bytes(g, colkind);
}

// The checks of one layer of an ADMM update (sadmm_admm_update and each item
// of sadmm_admm_update_batch).
static sadmm_status check_admm_item(const sadmm_conv_desc* d, const void* W, const void* U, const void* Z, int wdt,
                                    int k_filters, int colkind, int k_cols, const int* filt_idx, const int* col_idx,
                                    const double* keys_out, const void* workspace, size_t ws_bytes, Geometry* gout)
{
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    st = check_project_args(g, W, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out);
    if (st != SADMM_OK) return st;
    if (!U || !Z || !workspace) return SADMM_EINVAL;
    if (ws_bytes < admm_workspace_bytes(g, colkind)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0) return SADMM_EINVAL;
    const size_t esz = (wdt == SADMM_FP32) ? 4 : 2;
    const uintptr_t bytes = (uintptr_t)(g.f * g.k) * esz;
    const uintptr_t w = reinterpret_cast<uintptr_t>(W), u = reinterpret_cast<uintptr_t>(U),
                    z = reinterpret_cast<uintptr_t>(Z);
    if (((w | u | z) & (esz - 1)) != 0) return SADMM_EINVAL;
    auto overlap = [bytes](uintptr_t p, uintptr_t q) { return p < q + bytes && q < p + bytes; };
    if (overlap(w, u) || overlap(w, z) || overlap(u, z)) return SADMM_EINVAL;
    if (g.f > 65535) return SADMM_EUNSUPPORTED;
    *gout = g;
    return SADMM_OK;
}

sadmm_status sadmm_admm_update_batch(const sadmm_admm_item* items, int n, int wdt, void* stream)
{
    NvtxRange range("sadmm_admm_update_batch");
    if (!items || n < 1 || n > SADMM_MAX_BATCH) return SADMM_EINVAL;
    ProjItem pit[SADMM_MAX_BATCH];
    for (int l = 0; l < n; ++l) {
        const sadmm_admm_item& it = items[l];
        Geometry g;
        const sadmm_status st = check_admm_item(&it.desc, it.W, it.U, it.Z, wdt, it.k_filters, it.colkind, it.k_cols,
                                                it.filt_idx, it.col_idx, it.keys_out, it.workspace, it.ws_bytes, &g);
        if (st != SADMM_OK) return st;
        pit[l].g = g;
        pit[l].W = it.W;
        pit[l].U = it.U;
        pit[l].Z = it.Z;
        pit[l].k_filters = it.k_filters;
        pit[l].colkind = it.colkind;
        pit[l].k_cols = it.k_cols;
        pit[l].filt_idx = it.filt_idx;
        pit[l].col_idx = it.col_idx;
        pit[l].keys_out = it.keys_out;
        pit[l].ws = it.workspace;
        pit[l].rkeep = nullptr;
        pit[l].ckeep = nullptr;
    }
    return launch_admm_batch(pit, n, wdt, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_admm_update(const sadmm_conv_desc* d, const void* W, void* U, void* Z, int wdt, int k_filters,
                               int colkind, int k_cols, int* filt_idx, int* col_idx, double* keys_out,
                               void* workspace, size_t ws_bytes, void* stream)
{
    NvtxRange range("sadmm_admm_update");
    Geometry g;
    const sadmm_status st = check_admm_item(d, W, U, Z, wdt, k_filters, colkind, k_cols, filt_idx, col_idx,
                                            keys_out, workspace, ws_bytes, &g);
    if (st != SADMM_OK) return st;
    return launch_admm_update(g, W, U, Z, wdt, k_filters, colkind, k_cols, filt_idx, col_idx, keys_out,
                              workspace, static_cast<cudaStream_t>(stream));
}

size_t sadmm_elements_workspace_size(const sadmm_conv_desc* d)
{
    Geometry g;
    if (check_desc(d, &g) != SADMM_OK) return 0;
    return elements_workspace_bytes(g);
}

sadmm_status sadmm_project_elements(const sadmm_conv_desc* d, const void* W, const void* U, int wdt,
                                    long long k_elems, unsigned char* keep_out, void* workspace, size_t ws_bytes,
                                    void* stream)
{
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    if (!W || !keep_out || !workspace) return SADMM_EINVAL;
    if (wdt != SADMM_BF16 && wdt != SADMM_FP32) return SADMM_EINVAL;
    if (k_elems < 0 || k_elems > g.f * g.k) return SADMM_EINVAL;
    if (ws_bytes < elements_workspace_bytes(g)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0) return SADMM_EINVAL;
    const size_t esz = (wdt == SADMM_FP32) ? 4 : 2;
    if (((reinterpret_cast<uintptr_t>(W) | reinterpret_cast<uintptr_t>(U)) & (esz - 1)) != 0) return SADMM_EINVAL;
    return launch_elements(g, W, const_cast<void*>(U), nullptr, wdt, k_elems, keep_out, workspace,
                           static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_admm_update_elements(const sadmm_conv_desc* d, const void* W, void* U, void* Z, int wdt,
                                        long long k_elems, void* workspace, size_t ws_bytes, void* stream)
{
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    if (!W || !U || !Z || !workspace) return SADMM_EINVAL;
    if (wdt != SADMM_BF16 && wdt != SADMM_FP32) return SADMM_EINVAL;
    if (k_elems < 0 || k_elems > g.f * g.k) return SADMM_EINVAL;
    if (ws_bytes < elements_workspace_bytes(g)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255) != 0) return SADMM_EINVAL;
    const size_t esz = (wdt == SADMM_FP32) ? 4 : 2;
    const uintptr_t bytes = (uintptr_t)(g.f * g.k) * esz;
    const uintptr_t w = reinterpret_cast<uintptr_t>(W), u = reinterpret_cast<uintptr_t>(U),
                    z = reinterpret_cast<uintptr_t>(Z);
    if (((w | u | z) & (esz - 1)) != 0) return SADMM_EINVAL;
    auto overlap = [bytes](uintptr_t p, uintptr_t q) { return p < q + bytes && q < p + bytes; };
    if (overlap(w, u) || overlap(w, z) || overlap(u, z)) return SADMM_EINVAL;
    return launch_elements(g, W, U, Z, wdt, k_elems, nullptr, workspace, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_plan_init(sadmm_plan* plan, const sadmm_conv_desc* d, int n_filt, int colkind,
                             int n_colgroups)
{
    return sadmm_plan_init_ctas(plan, d, n_filt, colkind, n_colgroups, 0);
}

sadmm_status sadmm_plan_init_ctas(sadmm_plan* plan, const sadmm_conv_desc* d, int n_filt, int colkind,
                                  int n_colgroups, int max_ctas)
{
    if (!plan || max_ctas < 0) return SADMM_EINVAL;
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    if (n_filt < 0 || n_filt > g.f) return SADMM_EINVAL;
    long long n_cols;
    if (colkind == SADMM_COL_SHAPE) {
        if (n_colgroups < 0 || n_colgroups > g.k) return SADMM_EINVAL;
        n_cols = n_colgroups;
    } else if (colkind == SADMM_COL_CHANNEL) {
        if (n_colgroups < 0 || n_colgroups > g.cg) return SADMM_EINVAL;
        n_cols = (long long)n_colgroups * g.taps;
    } else if (colkind == SADMM_COL_NONE) {
        n_colgroups = (int)g.k;
        n_cols = g.k;
    } else {
        return SADMM_EINVAL;
    }
    if (n_cols > 8192) return SADMM_EUNSUPPORTED;
    sadmm_plan p;
    memset(&p, 0, sizeof(p));
    p.desc = *d;
    p.ctas = device_sm_count();  // CTAs a forward launches at most (one per SM)
    if (max_ctas > 0 && max_ctas < p.ctas) p.ctas = max_ctas;
    p.n_filt = n_filt;
    p.colkind = colkind;
    p.n_colgroups = n_colgroups;
    p.n_cols = (int)n_cols;
    p.k_pad = (int)(n_cols < 64 ? 64 : round_up(n_cols, 64));
    // rows of the packed matrix per conv group: the most kept filters any group
    // can have, in tiles of at most 256 rows (multiples of 16)
    long long rmax = n_filt < g.fg ? n_filt : g.fg;
    if (rmax < 16) rmax = 16;
    rmax = round_up(rmax, 16);
    p.n_tiles = (int)((rmax + 255) / 256);
    p.bn = (int)round_up((rmax + p.n_tiles - 1) / p.n_tiles, 16);
    p.n_pad = p.bn * p.n_tiles;
    if (p.n_pad > 4096) return SADMM_EUNSUPPORTED;
    size_t off = 0;
    auto take = [&off](size_t bytes) {
        const size_t at = off;
        off += (size_t)round_up((long long)bytes, 1024);
        return at;
    };
    p.off_wp = take((size_t)g.groups * p.n_pad * p.k_pad * 2);
    p.off_gather = take((size_t)p.k_pad * 8 + (size_t)(p.k_pad / 64) * 8);  // entries + stage channel ranges
    p.off_colidx = take((size_t)p.k_pad * 4);
    p.off_rowmap = take((size_t)g.groups * p.n_pad * 4);
    p.off_zeromap = take((size_t)g.f * 4);
    p.off_counts = take((size_t)g.groups * 2 * 4);
    p.splits = 1;
    p.stages_per_split = p.k_pad / 64;
    // input-slab path: one conv group, every column of the kept channels kept,
    // few slab channels, one filter tile, more than one block tap (a 1 x 1
    // block kernel reads contiguous input rows, which the gathered path does
    // as fast without the space-to-depth pass), and a slab GEMM at most twice
    // as wide
    const bool cols_whole = colkind == SADMM_COL_NONE || colkind == SADMM_COL_CHANNEL ||
                            (colkind == SADMM_COL_SHAPE && n_cols == g.k);
    if (g.t == 1 && g.kt == 1 && g.groups == 1 && p.n_tiles == 1 && cols_whole && n_cols > 0) {
        const long long nck = colkind == SADMM_COL_CHANNEL ? n_colgroups : g.c;
        const long long R = (g.kh + g.sh - 1) / g.sh, Q = (g.kw + g.sw - 1) / g.sw;
        const long long cs = round_up(nck * g.sh * g.sw, 16);
        const long long hb = g.oh + R - 1, wb = g.ow + Q - 1;
        const long long pimg = round_up(hb * wb, 8);
        const long long sp = round_up(128 + (R - 1) * wb + (Q - 1), 8);
        const long long kpad_s = round_up(R * Q * cs, 64);
        const long long xs_bytes = g.n * cs * pimg * 2;
        if (R * Q >= 2 && cs <= 64 && sp / 8 <= 256 && kpad_s <= 2 * p.k_pad && pimg < (1ll << 28) && hb <= 65535 && g.n <= 65535 &&
            xs_bytes <= (4ll << 30) && slab_stages(p.bn, (int)kpad_s, (int)cs, (int)sp) >= 2) {
            p.xs_mode = 1;
            p.xs_r = (int)R;
            p.xs_q = (int)Q;
            p.xs_cs = (int)cs;
            p.xs_hb = (int)hb;
            p.xs_wb = (int)wb;
            p.xs_pimg = (int)pimg;
            p.xs_sp = (int)sp;
            p.xs_kpad = (int)kpad_s;
            p.off_xs = take((size_t)xs_bytes);
            p.off_wps = take((size_t)p.bn * kpad_s * 2);
            p.off_scol = take((size_t)(kpad_s + cs) * 4);
        }
    }
    // split K' when the layer has fewer output tiles than the device has SMs
    if (!p.xs_mode) {
        const long long nks = p.k_pad / 64;
        const long long m_tiles = (g.m + 127) / 128;
        const long long upairs = (p.n_tiles + (p.n_tiles >= 2 ? 1 : 0)) / (p.n_tiles >= 2 ? 2 : 1);
        const long long units = m_tiles * g.groups * upairs;
        const long long sms = p.ctas;
        const long long rows = g.groups * p.n_pad + g.groups * g.fg;  // finalize rows
        if (units < sms && nks >= 2 && rows <= 65535) {
            long long want = (sms + units - 1) / units;
            if (want > nks) want = nks;
            long long ksps = (nks + want - 1) / want;
            // a split of a short K' (at most 8 stages) carries at least two
            // stages: a one-stage split pays a whole prologue and a partial-sum
            // round trip for one stage of work (measured slower on GB300)
            if (nks <= 8 && ksps < 2) ksps = 2;
            const long long splits = (nks + ksps - 1) / ksps;
            const long long bytes = splits * g.groups * p.n_pad * m_tiles * 128 * 4;
            if (splits > 1 && bytes <= (256ll << 20)) {
                p.splits = (int)splits;
                p.stages_per_split = (int)ksps;
                p.off_partial = take((size_t)bytes);
            }
        }
        // stream-K when the tiles do not spread evenly: a run of L stages per
        // CTA instead of ceil(units / sms) whole tiles, if that shortens the
        // busiest CTA by at least 1/8 and no tile is cut more than once
        // (L >= nks).  A cut tile costs a write and a read of 8 bytes per pixel
        // and filter row; measured on GB300 that pays only with two TMEM
        // accumulator sets (the finishing piece overlaps the next tile's MMAs)
        // and a K' of at least four times the filter rows.
        const long long total = units * nks;
        const int nacc = p.n_tiles >= 2 ? 2 : 1;
        const bool two_acc = 2 * nacc * round_up(p.bn, 32) <= 512;
        if (p.splits == 1 && units >= sms && two_acc && p.k_pad >= 4ll * p.bn &&
            total < (1ll << 31) - (1ll << 20)) {
            const long long dp = (units + sms - 1) / sms * nks;
            const long long L = (total + sms - 1) / sms;
            if (L >= nks && (dp - L) * 8 >= dp) {
                const long long grid = (total + L - 1) / L;
                const long long cols = (long long)nacc * p.bn;
                // arrival counters, then the partial sums [slot][2][cols][128 pixels]
                const long long bytes = round_up(grid * 4, 1024) + grid * 2 * cols * 128 * 4;
                if (bytes <= (256ll << 20)) {
                    p.sk_len = (int)L;
                    p.sk_grid = (int)grid;
                    p.off_sk = take((size_t)bytes);
                }
            }
        }
    }
    p.dev_bytes = off;
    p.dev = nullptr;
    *plan = p;
    return SADMM_OK;
}

namespace {

// The host checks of one layer of sadmm_pack / sadmm_pack_batch.
sadmm_status check_pack(const sadmm_plan* plan, const void* W, int wdt, const int* filt_idx, const int* col_idx,
                        const void* dev, size_t dev_bytes, Geometry* g)
{
    if (!plan || !W || !dev) return SADMM_EINVAL;
    sadmm_status st = check_desc(&plan->desc, g);
    if (st != SADMM_OK) return st;
    if (wdt != SADMM_BF16 && wdt != SADMM_FP32) return SADMM_EINVAL;
    if (dev_bytes < plan->dev_bytes) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(dev) & 255) != 0) return SADMM_EINVAL;
    if (plan->n_filt < (int)g->f && plan->n_filt > 0 && !filt_idx) return SADMM_EINVAL;
    if (plan->colkind != SADMM_COL_NONE && plan->n_colgroups > 0 && !col_idx) return SADMM_EINVAL;
    return SADMM_OK;
}

}  // namespace

sadmm_status sadmm_pack(sadmm_plan* plan, const void* W, int wdt, const int* filt_idx, const int* col_idx,
                        void* dev, size_t dev_bytes, void* stream)
{
    NvtxRange range("sadmm_pack");
    PackJob job;
    sadmm_status st = check_pack(plan, W, wdt, filt_idx, col_idx, dev, dev_bytes, &job.g);
    if (st != SADMM_OK) return st;
    if (device_cc_major() < 10) return SADMM_EUNSUPPORTED;
    plan->dev = dev;
    job.plan = plan;
    job.W = W;
    job.filt_idx = filt_idx;
    job.col_idx = col_idx;
    return launch_pack_batch(&job, 1, wdt, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_pack_batch(sadmm_pack_item* items, int n, int wdt, void* stream)
{
    NvtxRange range("sadmm_pack_batch");
    if (!items || n < 1 || n > SADMM_MAX_BATCH) return SADMM_EINVAL;
    PackJob jobs[SADMM_MAX_BATCH];
    for (int i = 0; i < n; ++i) {
        const sadmm_pack_item& it = items[i];
        sadmm_status st = check_pack(it.plan, it.W, wdt, it.filt_idx, it.col_idx, it.dev, it.dev_bytes, &jobs[i].g);
        if (st != SADMM_OK) return st;
        for (int j = 0; j < i; ++j)
            if (items[j].plan == it.plan) return SADMM_EINVAL;  // one plan per item
        jobs[i].plan = it.plan;
        jobs[i].W = it.W;
        jobs[i].filt_idx = it.filt_idx;
        jobs[i].col_idx = it.col_idx;
    }
    if (device_cc_major() < 10) return SADMM_EUNSUPPORTED;
    for (int i = 0; i < n; ++i) items[i].plan->dev = items[i].dev;
    return launch_pack_batch(jobs, n, wdt, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_conv_fwd_phase(const sadmm_plan* plan, const void* x, const float* bias, int relu, void* y,
                                  int ydt, int phase, void* stream)
{
    NvtxRange range("sadmm_conv_fwd");
    if (!plan || !plan->dev) return SADMM_EINVAL;
    if (phase != SADMM_FWD_ALL && phase != SADMM_FWD_INPUT && phase != SADMM_FWD_REST) return SADMM_EINVAL;
    const bool needs_x = phase != SADMM_FWD_REST || !plan->xs_mode;  // the rest of a slab plan reads its copy
    const bool needs_y = phase != SADMM_FWD_INPUT;
    if ((needs_x && !x) || (needs_y && !y)) return SADMM_EINVAL;
    Geometry g;
    sadmm_status st = check_desc(&plan->desc, &g);
    if (st != SADMM_OK) return st;
    if (needs_y && ydt != SADMM_BF16 && ydt != SADMM_FP32) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(x) & 1) != 0) return SADMM_EINVAL;
    if (needs_y && (reinterpret_cast<uintptr_t>(y) & (ydt == SADMM_FP32 ? 3 : 1)) != 0) return SADMM_EINVAL;
    if (bias && (reinterpret_cast<uintptr_t>(bias) & 3) != 0) return SADMM_EINVAL;
    if (device_cc_major() < 10) return SADMM_EUNSUPPORTED;
    return launch_conv_fwd(plan, g, x, bias, relu, y, ydt, phase, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_conv_fwd(const sadmm_plan* plan, const void* x, const float* bias, int relu, void* y,
                            int ydt, void* stream)
{
    return sadmm_conv_fwd_phase(plan, x, bias, relu, y, ydt, SADMM_FWD_ALL, stream);
}

size_t sadmm_conv_bwd_workspace_size(const sadmm_plan* plan)
{
    if (!plan) return 0;
    Geometry g;
    if (check_desc(&plan->desc, &g) != SADMM_OK) return 0;
    return bwd_workspace_bytes(plan, g);
}

size_t sadmm_conv_bwd_workspace_size_chunk(const sadmm_plan* plan, long long chunk_pixels)
{
    if (!plan || chunk_pixels < 1) return 0;
    Geometry g;
    if (check_desc(&plan->desc, &g) != SADMM_OK) return 0;
    return bwd_workspace_bytes(plan, g, chunk_pixels);
}

sadmm_status sadmm_conv_bwd(const sadmm_plan* plan, const void* x, const void* dy, const void* y, int ydt, int relu,
                            float* dW, float* db, float* dx, void* workspace, size_t ws_bytes, void* stream)
{
    if (!plan || !plan->dev || !dy || !workspace) return SADMM_EINVAL;
    Geometry g;
    sadmm_status st = check_desc(&plan->desc, &g);
    if (st != SADMM_OK) return st;
    if (dW && !x) return SADMM_EINVAL;
    if (relu && !y) return SADMM_EINVAL;
    if (relu && ydt != SADMM_BF16 && ydt != SADMM_FP32) return SADMM_EINVAL;
    if (ws_bytes < bwd_workspace_bytes(plan, g, 256)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 1023) != 0) return SADMM_EINVAL;
    if (((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(dy)) & 1) != 0) return SADMM_EINVAL;
    if (((reinterpret_cast<uintptr_t>(dW) | reinterpret_cast<uintptr_t>(db) | reinterpret_cast<uintptr_t>(dx)) & 3) != 0)
        return SADMM_EINVAL;
    if (device_cc_major() < 10) return SADMM_EUNSUPPORTED;
    return launch_conv_bwd(plan, g, x, dy, y, ydt, relu, dW, db, dx, workspace, ws_bytes,
                           static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_gemm_bf16(const void* A, const void* B, float* C, long long M, long long N, long long K,
                             long long ldc, int accumulate, void* stream)
{
    if (!A || !B || !C) return SADMM_EINVAL;
    if (((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B) | reinterpret_cast<uintptr_t>(C)) & 15) != 0)
        return SADMM_EINVAL;
    int bn = 256;
    while (bn >= 16 && N % bn != 0) bn -= 16;
    if (bn < 16) return SADMM_EINVAL;
    if (device_cc_major() < 10) return SADMM_EUNSUPPORTED;
    return launch_gemm(A, B, C, M, N, K, ldc, bn, accumulate != 0, static_cast<cudaStream_t>(stream));
}

size_t sadmm_sparse_plan_size(const sadmm_conv_desc* d, long long capacity)
{
    Geometry g;
    if (check_desc(d, &g) != SADMM_OK) return 0;
    if (capacity < 0 || capacity > g.f * g.k) return 0;
    return sparse_plan_bytes(g, capacity);
}

sadmm_status sadmm_sparse_pack(const sadmm_conv_desc* d, const void* W, int wdt, const unsigned char* keep,
                               long long capacity, void* plan, size_t plan_bytes, void* stream)
{
    NvtxRange range("sadmm_sparse_pack");
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    if (!W || !keep || !plan) return SADMM_EINVAL;
    if (wdt != SADMM_BF16 && wdt != SADMM_FP32) return SADMM_EINVAL;
    if (capacity < 0 || capacity > g.f * g.k) return SADMM_EINVAL;
    if (plan_bytes < sparse_plan_bytes(g, capacity)) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(plan) & 255) != 0) return SADMM_EINVAL;
    if (g.f > 65535) return SADMM_EUNSUPPORTED;
    return launch_sparse_pack(g, W, wdt, keep, plan, capacity, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_sparse_conv_fwd(const sadmm_conv_desc* d, const void* plan, const void* x, const float* bias,
                                   int relu, void* y, int ydt, void* stream)
{
    NvtxRange range("sadmm_sparse_conv_fwd");
    Geometry g;
    sadmm_status st = check_desc(d, &g);
    if (st != SADMM_OK) return st;
    if (!plan || !x || !y) return SADMM_EINVAL;
    if (ydt != SADMM_BF16 && ydt != SADMM_FP32) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(plan) & 255) != 0 || (reinterpret_cast<uintptr_t>(x) & 1) != 0) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(y) & (ydt == SADMM_FP32 ? 3 : 1)) != 0) return SADMM_EINVAL;
    if (bias && (reinterpret_cast<uintptr_t>(bias) & 3) != 0) return SADMM_EINVAL;
    return launch_sparse_conv(g, plan, x, bias, relu, y, ydt, static_cast<cudaStream_t>(stream));
}

sadmm_status sadmm_selftest_wait(unsigned int limit_us, int arrive, int* result, void* stream)
{
    if (limit_us < 1 || limit_us > 1000000) return SADMM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(result) & 3) != 0) return SADMM_EINVAL;
    int* status = device_status_ptr();
    if (!status) return SADMM_ECUDA;
    k_selftest_wait<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(status, 1000ull * limit_us, arrive ? 1 : 0,
                                                                     result);
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

sadmm_status sadmm_last_device_status(void* stream)
{
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return SADMM_ECUDA;
    int v = 0;
    if (cudaMemcpyFromSymbol(&v, g_status_word, sizeof(int)) != cudaSuccess) return SADMM_ECUDA;
    if (v != 0) {
        const int zero = 0;
        cudaMemcpyToSymbol(g_status_word, &zero, sizeof(int));
    }
    if (v == kDevTimeout) return SADMM_ETIMEOUT;
    if (v == kDevBounds) return SADMM_EBOUNDS;
    if (v != 0) return SADMM_EINVAL;
    return SADMM_OK;
}

}  // extern "C"
