// elements.cu -- non-structured projection (Sec. 4, the solution of the
// Z-subproblem for non-structured sparsity: keep the gamma entries of
// V = W (+U) with the largest magnitudes, zero the rest), on its own and as
// the ADMM Z- and U-update.
//
// Keys are |V_e| with V formed exactly in fp64 (W + U of bf16 or fp32 values);
// as non-negative doubles their bit patterns order like the values.  The
// exact gamma-th largest key T is found by a most-significant-digit radix
// select over the 63 key bits (digits of 11, 11, 11, 11, 11 and 8 bits):
//   k_elem_hist   grid-stride pass: per-block shared histogram of the digit of
//                 every key that matches the prefix found so far, added to a
//                 global histogram.
//   k_elem_pick   one block: the digit at which the running count from the top
//                 reaches the remaining rank; extends the prefix, clears the
//                 histogram for the next pass.
// The passes stop early once the digit's bucket holds exactly the keys still
// needed: all of them are kept, the lower digits cannot change the choice, and
// keys are compared on the digits examined so far (T below is then the prefix).
// Entries with key > T are kept, and of the entries with key == T the ones
// with the lowest flat index e = a*K + j (ties to the lower index):
//   k_elem_eq     per chunk of kChunk consecutive entries: how many equal T.
//   k_elem_scan   one block: exclusive prefix of those counts over chunks.
//   k_elem_apply  per chunk: keep flags (and, for the ADMM update, Z and U).
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace sadmm {
namespace {

constexpr int kHistBins = 2048;
constexpr int kHistThreads = 512;
constexpr int kChunk = 4096;  // entries per chunk of the tie ranking
constexpr int kChunkThreads = 256;
// digit of pass p: bits [shift, shift + bits) of the key
SADMM_DEV int pass_shift(int p) { return p < 5 ? 52 - 11 * p : 0; }
SADMM_DEV int pass_bits(int p) { return p < 5 ? 11 : 8; }

struct SelState {
    unsigned long long prefix;  // key bits fixed so far
    unsigned long long mask;    // which bits the prefix fixes
    long long kk;               // rank still to find among keys matching the prefix
    int done;                   // 1: the choice is made (no further passes)
};

template <typename T>
SADMM_DEV double to_f64(T v);
template <>
SADMM_DEV double to_f64<__nv_bfloat16>(__nv_bfloat16 v) { return (double)__bfloat162float(v); }
template <>
SADMM_DEV double to_f64<float>(float v) { return (double)v; }

template <typename T>
SADMM_DEV T zero_of();
template <>
SADMM_DEV float zero_of<float>() { return 0.0f; }
template <>
SADMM_DEV __nv_bfloat16 zero_of<__nv_bfloat16>() { return __float2bfloat16_rn(0.0f); }

// State before the passes: rank k among all keys (prefix and mask empty),
// histogram cleared.  k <= 0 keeps nothing (a threshold above every key, no
// equals taken); k >= N keeps everything (threshold 0, every equal taken); the
// chunk offsets of the tie ranking are then zero.
__global__ void __launch_bounds__(256) k_elem_init(SelState* st, unsigned int* hist, unsigned int* eq_count,
                                                   long long nchunks, long long k, long long N)
{
    pdl_wait();  // after the kernel before it in the stream
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        if (k <= 0) *st = SelState{~0ull, ~0ull, 0, 1};
        else if (k >= N) *st = SelState{0ull, ~0ull, N, 1};
        else *st = SelState{0ull, 0ull, k, 0};
    }
    for (int i = blockIdx.x * 256 + threadIdx.x; i < kHistBins; i += gridDim.x * 256) hist[i] = 0u;
    if (k <= 0 || k >= N)
        for (long long i = blockIdx.x * 256 + threadIdx.x; i < nchunks; i += (long long)gridDim.x * 256)
            eq_count[i] = 0u;
}

template <typename T>
SADMM_DEV unsigned long long elem_key(const T* __restrict__ W, const T* __restrict__ U, long long e)
{
    double v = to_f64<T>(W[e]);
    if (U) v += to_f64<T>(U[e]);
    return (unsigned long long)__double_as_longlong(fabs(v));
}

template <typename T>
__global__ void __launch_bounds__(kHistThreads) k_elem_hist(const T* __restrict__ W, const T* __restrict__ U,
                                                            long long N, int pass, const SelState* __restrict__ st,
                                                            unsigned int* __restrict__ hist)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ unsigned int h[kHistBins];
    if (st->done) return;
    for (int i = threadIdx.x; i < kHistBins; i += kHistThreads) h[i] = 0u;
    __syncthreads();
    const unsigned long long prefix = st->prefix, mask = st->mask;
    const int shift = pass_shift(pass);
    const unsigned dmask = (1u << pass_bits(pass)) - 1u;
    for (long long e = (long long)blockIdx.x * kHistThreads + threadIdx.x; e < N;
         e += (long long)gridDim.x * kHistThreads) {
        const unsigned long long u = elem_key(W, U, e);
        if ((u & mask) == prefix) atomicAdd(&h[(unsigned)(u >> shift) & dmask], 1u);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kHistBins; i += kHistThreads)
        if (h[i]) atomicAdd(&hist[i], h[i]);
}

// One block of 1024 threads, two bins per thread.
__global__ void __launch_bounds__(1024) k_elem_pick(int pass, SelState* st, unsigned int* hist)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ unsigned long long s_tot[1024];
    if (st->done) return;
    const int tid = threadIdx.x;
    const int nb = 1 << pass_bits(pass);
    // bins in descending digit order: position q holds digit nb-1-q
    const int q0 = 2 * tid, q1 = 2 * tid + 1;
    const unsigned c0 = q0 < nb ? hist[nb - 1 - q0] : 0u;
    const unsigned c1 = q1 < nb ? hist[nb - 1 - q1] : 0u;
    s_tot[tid] = (unsigned long long)c0 + c1;
    __syncthreads();
    // inclusive prefix over threads (Hillis-Steele, fixed order)
    for (int o = 1; o < 1024; o <<= 1) {
        const unsigned long long v = tid >= o ? s_tot[tid - o] : 0ull;
        __syncthreads();
        s_tot[tid] += v;
        __syncthreads();
    }
    const unsigned long long before = tid > 0 ? s_tot[tid - 1] : 0ull;  // keys with a higher digit
    const long long kk = st->kk;
    __syncthreads();
    if (before < (unsigned long long)kk && (unsigned long long)kk <= s_tot[tid]) {
        const int shift = pass_shift(pass);
        int q = q0;
        unsigned long long cum = before;
        unsigned c = c0;
        if (cum + c0 < (unsigned long long)kk) { cum += c0; q = q1; c = c1; }
        const unsigned long long d = (unsigned long long)(nb - 1 - q);
        st->prefix |= d << shift;
        st->mask |= (unsigned long long)(nb - 1) << shift;
        st->kk = kk - (long long)cum;
        if ((unsigned long long)c == (unsigned long long)kk - cum) st->done = 1;  // the whole bucket is kept
    }
    // clear for the next pass (every block of this pass has finished)
    for (int i = tid; i < kHistBins; i += 1024) hist[i] = 0u;
}

template <typename T>
__global__ void __launch_bounds__(kChunkThreads) k_elem_eq(const T* __restrict__ W, const T* __restrict__ U,
                                                           long long N, const SelState* __restrict__ st,
                                                           unsigned int* __restrict__ eq_count)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ unsigned int s_n;
    if (threadIdx.x == 0) s_n = 0u;
    __syncthreads();
    const unsigned long long thr = st->prefix, mask = st->mask;
    const long long c0 = (long long)blockIdx.x * kChunk;
    unsigned n = 0;
    for (int i = threadIdx.x; i < kChunk; i += kChunkThreads) {
        const long long e = c0 + i;
        if (e < N && (elem_key(W, U, e) & mask) == thr) ++n;
    }
    if (n) atomicAdd(&s_n, n);
    __syncthreads();
    if (threadIdx.x == 0) eq_count[blockIdx.x] = s_n;
}

// Exclusive prefix of eq_count[0..nchunks) in place (one block, fixed order).
__global__ void __launch_bounds__(1024) k_elem_scan(unsigned int* eq_count, int nchunks)
{
    pdl_wait();  // after the kernel before it in the stream
    __shared__ unsigned int s[1024];
    __shared__ unsigned int carry;
    if (threadIdx.x == 0) carry = 0u;
    __syncthreads();
    for (int base = 0; base < nchunks; base += 1024) {
        const int i = base + threadIdx.x;
        const unsigned v = i < nchunks ? eq_count[i] : 0u;
        s[threadIdx.x] = v;
        __syncthreads();
        for (int o = 1; o < 1024; o <<= 1) {
            const unsigned t = threadIdx.x >= o ? s[threadIdx.x - o] : 0u;
            __syncthreads();
            s[threadIdx.x] += t;
            __syncthreads();
        }
        if (i < nchunks) eq_count[i] = carry + s[threadIdx.x] - v;
        __syncthreads();
        if (threadIdx.x == 0) carry += s[1023];
        __syncthreads();
    }
}

// Keep flags (keep_out) or the ADMM update (Z, U) of one chunk.  Equal keys
// are ranked in index order: the chunk's offset plus the ballot-prefix of the
// entries before them in the chunk.
template <typename T>
__global__ void __launch_bounds__(kChunkThreads) k_elem_apply(const T* __restrict__ W, T* __restrict__ U, T* Z,
                                                              long long N, const SelState* __restrict__ st,
                                                              const unsigned int* __restrict__ eq_off,
                                                              uint8_t* __restrict__ keep_out)
{
    pdl_wait();  // after the kernel before it in the stream
    const long long take_eq = st->kk;  // how many keys equal to the threshold are kept
    __shared__ unsigned int warp_n[kChunkThreads / 32];
    __shared__ unsigned int run;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned long long Tk = st->prefix, kmask = st->mask;
    if (threadIdx.x == 0) run = eq_off[blockIdx.x];
    __syncthreads();
    const long long c0 = (long long)blockIdx.x * kChunk;
    for (int base = 0; base < kChunk; base += kChunkThreads) {
        const long long e = c0 + base + threadIdx.x;
        const bool valid = e < N;
        T w = zero_of<T>(), u = zero_of<T>();
        unsigned long long key = 0ull;
        if (valid) {
            w = W[e];
            if (U) u = U[e];
            double v = to_f64<T>(w);
            if (U) v += to_f64<T>(u);
            key = (unsigned long long)__double_as_longlong(fabs(v)) & kmask;
        }
        const bool eq = valid && key == Tk;
        const unsigned b = __ballot_sync(0xffffffffu, eq);
        if (lane == 0) warp_n[warp] = __popc(b);
        __syncthreads();
        unsigned before = run;
        for (int q = 0; q < warp; ++q) before += warp_n[q];
        before += __popc(b & ((1u << lane) - 1u));
        const bool keep = valid && (key > Tk || (eq && (long long)before < take_eq));
        if (valid) {
            if (keep_out) keep_out[e] = keep ? 1 : 0;
            if (Z) {
                // V rounded once to T (as in the structured ADMM update)
                T vt;
                if constexpr (sizeof(T) == 4) {
                    vt = (T)((float)w + (float)u);
                } else {
                    vt = __float2bfloat16_rn(__bfloat162float(w) + __bfloat162float(u));
                }
                const T zero = zero_of<T>();
                Z[e] = keep ? vt : zero;
                U[e] = keep ? zero : vt;
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            unsigned t = 0;
            for (int q = 0; q < kChunkThreads / 32; ++q) t += warp_n[q];
            run += t;
        }
        __syncthreads();
    }
}

template <typename T>
sadmm_status run_elements(const Geometry& g, const T* W, T* U, T* Z, long long k, uint8_t* keep_out, void* ws,
                          cudaStream_t s)
{
    const long long N = g.f * g.k;
    char* base = static_cast<char*>(ws);
    SelState* st = reinterpret_cast<SelState*>(base);
    unsigned int* hist = reinterpret_cast<unsigned int*>(base + 256);
    unsigned int* eq_count = hist + kHistBins;
    const long long nchunks = (N + kChunk - 1) / kChunk;
    const unsigned init_blocks = (unsigned)std::min<long long>((nchunks + 255) / 256 + 1, 1024);
    launch_pdl(k_elem_init, dim3(init_blocks), dim3(256), 0, s, st, hist, eq_count, nchunks, k, N);
    if (k > 0 && k < N) {
        const int blocks = (int)std::min<long long>((N + kHistThreads - 1) / kHistThreads, 4LL * device_sm_count());
        for (int pass = 0; pass < 6; ++pass) {
            launch_pdl(k_elem_hist<T>, dim3(blocks), dim3(kHistThreads), 0, s, W, U, N, pass,
                       static_cast<const SelState*>(st), hist);
            launch_pdl(k_elem_pick, dim3(1), dim3(1024), 0, s, pass, st, hist);
        }
        launch_pdl(k_elem_eq<T>, dim3((unsigned)nchunks), dim3(kChunkThreads), 0, s, W, U, N,
                   static_cast<const SelState*>(st), eq_count);
        launch_pdl(k_elem_scan, dim3(1), dim3(1024), 0, s, eq_count, (int)nchunks);
    }
    launch_pdl(k_elem_apply<T>, dim3((unsigned)nchunks), dim3(kChunkThreads), 0, s, W, U, Z, N,
               static_cast<const SelState*>(st), static_cast<const unsigned int*>(eq_count), keep_out);
    return cudaGetLastError() == cudaSuccess ? SADMM_OK : SADMM_ECUDA;
}

}  // namespace

size_t elements_workspace_bytes(const Geometry& g)
{
    const long long N = g.f * g.k;
    return 256 + kHistBins * 4 + (size_t)((N + kChunk - 1) / kChunk) * 4 + 256;
}

sadmm_status launch_elements(const Geometry& g, const void* W, void* U, void* Z, int wdt, long long k,
                             uint8_t* keep_out, void* ws, cudaStream_t s)
{
    if (wdt == SADMM_BF16)
        return run_elements<__nv_bfloat16>(g, (const __nv_bfloat16*)W, (__nv_bfloat16*)U, (__nv_bfloat16*)Z, k,
                                           keep_out, ws, s);
    return run_elements<float>(g, (const float*)W, (float*)U, (float*)Z, k, keep_out, ws, s);
}

}  // namespace sadmm
