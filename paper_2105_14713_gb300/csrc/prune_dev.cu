// Device-side 1xN pruning and BSR packing: the same results as the host
// onexn_prune / onexn_pack, bit for bit, for weights that live on the GPU
// (a fine-tuning loop re-pruning or re-packing without a host round trip).
//
// Prune (Eq. 4 / Eq. 5 and the top-(1-p) solution after Eq. 5):
//   1. one thread per block: its l1 norm in fp64, summed in the order n,
//      then kh, kw (the host's order; additions only, so no contraction can
//      change a bit);
//   2. the keep-th largest norm T by a most-significant-digit radix select
//      over the norms' bit patterns (for non-negative doubles the unsigned
//      bit order is the numeric order): eight passes of an 8-bit histogram
//      over the blocks whose higher digits match, each followed by a
//      one-thread pick of the digit that holds the keep-th largest;
//   3. kept = norm > T, or norm == T and among the first k_rem such blocks
//      in index order (ties go to the lower block index g*nb + b): the rank
//      among the equal blocks comes from per-chunk counts, their exclusive
//      scan, and a block scan inside each chunk.
// Pack (Sec. 3.4): per col-group count of kept indices, an exclusive scan
// into P, then per group a block scan over k that places each kept index
// (increasing k) and its N weights (fp32 copy, or bf16 round-to-nearest-
// even) at I[z], D[z].
#include "conv_common.cuh"
#include "onexn_internal.h"

#include <cuda_bf16.h>

using onexn::fail;

namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 4 * kThreads;    // indices per CTA in the rank pass

struct SelState {
    unsigned long long prefix;   // digits of T decided so far
    unsigned long long pmask;    // which bits of prefix are decided
    long long k_rem;             // rank of T among the blocks matching prefix (from the top)
};

__device__ __forceinline__ double absw(const float *W, int64_t at) { return fabs(static_cast<double>(W[at])); }

__global__ void __launch_bounds__(kThreads)
score_kernel(const float *__restrict__ W, int C_in, int KH, int KW, int N, int gran, int64_t total,
             unsigned long long *__restrict__ key)
{
    const int K = KH * KW * C_in;
    const int nb = gran == ONEXN_GRAN_TAP ? K : C_in;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t g = i / nb;
        const int b = static_cast<int>(i - g * nb);
        double s = 0.0;
        if (gran == ONEXN_GRAN_TAP) {
            const int tap = b / C_in, c = b - (b / C_in) * C_in;
            for (int n = 0; n < N; ++n)
                s = __dadd_rn(s, absw(W, ((g * N + n) * C_in + c) * KH * KW + tap));
        } else {
            for (int n = 0; n < N; ++n)
                for (int t = 0; t < KH * KW; ++t)
                    s = __dadd_rn(s, absw(W, ((g * N + n) * C_in + b) * KH * KW + t));
        }
        key[i] = static_cast<unsigned long long>(__double_as_longlong(s));
    }
}

__global__ void sel_init_kernel(SelState *st, unsigned int *hist, long long keep)
{
    if (threadIdx.x == 0) {
        st->prefix = 0ull;
        st->pmask = 0ull;
        st->k_rem = keep;
    }
    hist[threadIdx.x] = 0u;
}

__global__ void __launch_bounds__(kThreads)
hist_kernel(const unsigned long long *__restrict__ key, int64_t total, const SelState *st, int shift,
            unsigned int *hist)
{
    __shared__ unsigned int h[256];
    h[threadIdx.x] = 0u;
    __syncthreads();
    const unsigned long long prefix = st->prefix, pmask = st->pmask;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const unsigned long long k = key[i];
        if ((k & pmask) == prefix) atomicAdd(&h[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (h[threadIdx.x]) atomicAdd(&hist[threadIdx.x], h[threadIdx.x]);
}

// One thread: the digit (from the top) whose bucket holds the k_rem-th
// largest of the matching keys; clears the histogram for the next pass.
__global__ void pick_kernel(SelState *st, unsigned int *hist, int shift)
{
    __shared__ int chosen;
    if (threadIdx.x == 0) {
        long long cum = 0;
        chosen = 0;
        for (int d = 255; d >= 0; --d) {
            const long long c = hist[d];
            if (cum + c >= st->k_rem) {
                chosen = d;
                break;
            }
            cum += c;
        }
        st->k_rem -= cum;
        st->prefix |= static_cast<unsigned long long>(chosen) << shift;
        st->pmask |= 255ull << shift;
    }
    __syncthreads();
    hist[threadIdx.x] = 0u;
}

// Blocks equal to T per chunk of kChunk indices.
__global__ void __launch_bounds__(kThreads)
eq_count_kernel(const unsigned long long *__restrict__ key, int64_t total, const SelState *st,
                unsigned int *chunk_cnt)
{
    __shared__ unsigned int c;
    if (threadIdx.x == 0) c = 0u;
    __syncthreads();
    const unsigned long long T = st->prefix;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kChunk;
    unsigned int mine = 0;
    for (int j = 0; j < 4; ++j) {
        const int64_t i = base + threadIdx.x * 4 + j;
        if (i < total && key[i] == T) ++mine;
    }
    if (mine) atomicAdd(&c, mine);
    __syncthreads();
    if (threadIdx.x == 0) chunk_cnt[blockIdx.x] = c;
}

// Exclusive scan of n counts in place, by one CTA (serial over blocks of
// kThreads, a warp-shuffle scan inside each).
__device__ unsigned long long block_exclusive_scan(unsigned int v, unsigned long long *total_out)
{
    __shared__ unsigned long long warp_tot[kThreads / 32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    unsigned long long x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[w] = x;
    __syncthreads();
    unsigned long long before = 0, all = 0;
    for (int i = 0; i < kThreads / 32; ++i) {
        if (i < w) before += warp_tot[i];
        all += warp_tot[i];
    }
    __syncthreads();
    *total_out = all;
    return before + x - v;
}

__global__ void __launch_bounds__(kThreads) scan_u32_kernel(unsigned int *a, int64_t n)
{
    unsigned long long run = 0;
    for (int64_t b = 0; b < n; b += kThreads) {
        const int64_t i = b + threadIdx.x;
        const unsigned int v = i < n ? a[i] : 0u;
        unsigned long long tot;
        const unsigned long long ex = block_exclusive_scan(v, &tot);
        if (i < n) a[i] = static_cast<unsigned int>(run + ex);
        run += tot;
    }
}

__global__ void __launch_bounds__(kThreads)
mark_kernel(const unsigned long long *__restrict__ key, int64_t total, const SelState *st,
            const unsigned int *chunk_off, int gran, int C_in, int taps, int K, uint8_t *__restrict__ mask)
{
    const unsigned long long T = st->prefix;
    const long long k_rem = st->k_rem;
    const int64_t base = static_cast<int64_t>(blockIdx.x) * kChunk + threadIdx.x * 4;
    unsigned int eq = 0;
    bool gt[4], is_eq[4];
    for (int j = 0; j < 4; ++j) {
        const int64_t i = base + j;
        const unsigned long long k = i < total ? key[i] : 0ull;
        gt[j] = i < total && k > T;
        is_eq[j] = i < total && k == T;
        eq += is_eq[j] ? 1u : 0u;
    }
    unsigned long long tot;
    unsigned long long rank = chunk_off[blockIdx.x] + block_exclusive_scan(eq, &tot);
    for (int j = 0; j < 4; ++j) {
        const int64_t i = base + j;
        if (i >= total) break;
        bool keep = gt[j];
        if (is_eq[j]) {
            keep = static_cast<long long>(rank) < k_rem;
            ++rank;
        }
        const uint8_t m = keep ? 1 : 0;
        if (gran == ONEXN_GRAN_TAP) {
            mask[i] = m;
        } else {
            const int64_t g = i / C_in;
            const int c = static_cast<int>(i - g * C_in);
            for (int t = 0; t < taps; ++t) mask[g * K + static_cast<int64_t>(t) * C_in + c] = m;
        }
    }
}

__global__ void fill_u8_kernel(uint8_t *p, int64_t n, uint8_t v)
{
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        p[i] = v;
}

// ---- pack ----
__global__ void __launch_bounds__(kThreads) pack_count_kernel(const uint8_t *__restrict__ mask, int K,
                                                              unsigned int *cnt)
{
    const uint8_t *m = mask + static_cast<int64_t>(blockIdx.x) * K;
    unsigned int c = 0;
    for (int k = threadIdx.x; k < K; k += kThreads) c += m[k] ? 1u : 0u;
    unsigned long long tot;
    block_exclusive_scan(c, &tot);
    if (threadIdx.x == 0) cnt[blockIdx.x] = static_cast<unsigned int>(tot);
}

__global__ void __launch_bounds__(kThreads) pack_p_kernel(const unsigned int *cnt, int G, int32_t *P)
{
    unsigned long long run = 0;
    for (int b = 0; b < G; b += kThreads) {
        const int g = b + threadIdx.x;
        const unsigned int v = g < G ? cnt[g] : 0u;
        unsigned long long tot;
        const unsigned long long ex = block_exclusive_scan(v, &tot);
        if (g < G) P[g] = static_cast<int32_t>(run + ex);
        run += tot;
    }
    if (threadIdx.x == 0) P[G] = static_cast<int32_t>(run);
}

template <bool kBf16>
__global__ void __launch_bounds__(kThreads)
pack_fill_kernel(const float *__restrict__ W, const uint8_t *__restrict__ mask, int C_in, int KH, int KW, int N,
                 const int32_t *__restrict__ P, int32_t *__restrict__ I, void *__restrict__ D, int64_t t_cap)
{
    const int g = blockIdx.x;
    const int K = KH * KW * C_in;
    const uint8_t *m = mask + static_cast<int64_t>(g) * K;
    int64_t z0 = P[g];
    for (int k0 = 0; k0 < K; k0 += kThreads) {
        const int k = k0 + threadIdx.x;
        const bool kept = k < K && m[k] != 0;
        unsigned long long tot;
        const unsigned long long pos = block_exclusive_scan(kept ? 1u : 0u, &tot);
        const int64_t z = z0 + static_cast<int64_t>(pos);
        if (kept && z < t_cap) {
            I[z] = k;
            const int tap = k / C_in, c = k - (k / C_in) * C_in;
            for (int n = 0; n < N; ++n) {
                const float v = W[((static_cast<int64_t>(g) * N + n) * C_in + c) * KH * KW + tap];
                if (kBf16)
                    static_cast<__nv_bfloat16 *>(D)[z * N + n] = __float2bfloat16_rn(v);
                else
                    static_cast<float *>(D)[z * N + n] = v;
            }
        }
        z0 += static_cast<int64_t>(tot);
    }
}

bool dims_ok(int C_out, int C_in, int KH, int KW)
{
    return C_out > 0 && C_in > 0 && KH > 0 && KW > 0 &&
           static_cast<int64_t>(C_out) * KH * KW * C_in < (int64_t(1) << 31);
}

int grid_for(int64_t n, int sms)
{
    const int64_t b = (n + kThreads - 1) / kThreads;
    const int64_t cap = static_cast<int64_t>(sms) * 8;
    return static_cast<int>(b < 1 ? 1 : b < cap ? b : cap);
}

size_t align256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

struct PruneWs {
    size_t keys, state, hist, chunks, total;
};

PruneWs prune_ws_layout(int64_t nblocks)
{
    PruneWs w{};
    const int64_t n_chunks = (nblocks + kChunk - 1) / kChunk;
    w.keys = 0;
    w.state = align256(static_cast<size_t>(nblocks) * 8);
    w.hist = w.state + 256;
    w.chunks = w.hist + 256 * 4;
    w.total = align256(w.chunks + static_cast<size_t>(n_chunks) * 4);
    return w;
}

}  // namespace

extern "C" onexn_status onexn_prune_device_workspace_size(int C_out, int C_in, int KH, int KW, int N, int gran,
                                                          size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "prune_device: bytes is NULL");
    if (!dims_ok(C_out, C_in, KH, KW)) return fail(ONEXN_EINVAL, "prune_device: bad dimensions");
    if (N < 1 || C_out % N) return fail(ONEXN_EINVAL, "prune_device: N=%d must divide C_out=%d", N, C_out);
    if (gran != ONEXN_GRAN_TAP && gran != ONEXN_GRAN_KERNEL)
        return fail(ONEXN_EINVAL, "prune_device: unknown granularity %d", gran);
    const int64_t G = C_out / N;
    const int64_t nb = gran == ONEXN_GRAN_TAP ? static_cast<int64_t>(KH) * KW * C_in : C_in;
    *bytes = prune_ws_layout(G * nb).total;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_prune_device(const float *W, int C_out, int C_in, int KH, int KW, int N, double rate,
                                           int gran, uint8_t *mask, int64_t *kept, void *workspace,
                                           size_t workspace_bytes, void *stream)
{
    onexn::clear_error();
    size_t need = 0;
    onexn_status st = onexn_prune_device_workspace_size(C_out, C_in, KH, KW, N, gran, &need);
    if (st != ONEXN_OK) return st;
    if (!W || !mask || !kept) return fail(ONEXN_EINVAL, "prune_device: NULL pointer");
    if (!(rate >= 0.0 && rate <= 1.0)) return fail(ONEXN_EINVAL, "prune_device: rate %g outside [0, 1]", rate);
    if (!workspace || workspace_bytes < need)
        return fail(ONEXN_EINVAL, "prune_device: needs %zu bytes of workspace, got %zu", need, workspace_bytes);
    if (reinterpret_cast<uintptr_t>(workspace) & 255u)
        return fail(ONEXN_EINVAL, "prune_device: workspace must be 256-byte aligned");
    const int G = C_out / N, K = KH * KW * C_in;
    const int64_t nb = gran == ONEXN_GRAN_TAP ? K : C_in;
    const int64_t total = static_cast<int64_t>(G) * nb;
    int64_t keep = 0;
    st = onexn_keep_count(total, rate, &keep);
    if (st != ONEXN_OK) return st;
    *kept = keep;
    int sms = 0;
    cudaError_t e = onexn::device_sm_count(&sms);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "prune_device: %s", cudaGetErrorString(e));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t mask_n = static_cast<int64_t>(G) * K;
    if (keep == 0 || keep == total) {
        fill_u8_kernel<<<grid_for(mask_n, sms), kThreads, 0, s>>>(mask, mask_n, keep ? 1 : 0);
    } else {
        const PruneWs L = prune_ws_layout(total);
        unsigned char *ws = static_cast<unsigned char *>(workspace);
        auto *key = reinterpret_cast<unsigned long long *>(ws + L.keys);
        auto *sel = reinterpret_cast<SelState *>(ws + L.state);
        auto *hist = reinterpret_cast<unsigned int *>(ws + L.hist);
        auto *chunk = reinterpret_cast<unsigned int *>(ws + L.chunks);
        const int grid = grid_for(total, sms);
        score_kernel<<<grid, kThreads, 0, s>>>(W, C_in, KH, KW, N, gran, total, key);
        sel_init_kernel<<<1, 256, 0, s>>>(sel, hist, keep);
        for (int shift = 56; shift >= 0; shift -= 8) {
            hist_kernel<<<grid, kThreads, 0, s>>>(key, total, sel, shift, hist);
            pick_kernel<<<1, 256, 0, s>>>(sel, hist, shift);
        }
        const int64_t n_chunks = (total + kChunk - 1) / kChunk;
        eq_count_kernel<<<static_cast<unsigned>(n_chunks), kThreads, 0, s>>>(key, total, sel, chunk);
        scan_u32_kernel<<<1, kThreads, 0, s>>>(chunk, n_chunks);
        mark_kernel<<<static_cast<unsigned>(n_chunks), kThreads, 0, s>>>(key, total, sel, chunk, gran, C_in,
                                                                          KH * KW, K, mask);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "prune_device: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}

extern "C" onexn_status onexn_pack_device_workspace_size(int C_out, int N, size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "pack_device: bytes is NULL");
    if (C_out < 1 || N < 1 || C_out % N) return fail(ONEXN_EINVAL, "pack_device: N=%d must divide C_out=%d", N, C_out);
    *bytes = align256(static_cast<size_t>(C_out / N) * 4);
    return ONEXN_OK;
}

extern "C" onexn_status onexn_pack_device(const float *W, const uint8_t *mask, int C_out, int C_in, int KH, int KW,
                                          int N, int wdtype, int32_t *P, int32_t *I, void *D, int64_t t_cap,
                                          void *workspace, size_t workspace_bytes, void *stream)
{
    onexn::clear_error();
    if (!W || !mask || !P) return fail(ONEXN_EINVAL, "pack_device: NULL pointer");
    if (!dims_ok(C_out, C_in, KH, KW)) return fail(ONEXN_EINVAL, "pack_device: bad dimensions");
    if (N < 1 || C_out % N) return fail(ONEXN_EINVAL, "pack_device: N=%d must divide C_out=%d", N, C_out);
    if (wdtype != ONEXN_F32 && wdtype != ONEXN_BF16)
        return fail(ONEXN_EINVAL, "pack_device: unknown weight dtype %d", wdtype);
    if (t_cap < 0 || (t_cap > 0 && (!I || !D))) return fail(ONEXN_EINVAL, "pack_device: t_cap > 0 needs I and D");
    size_t need = 0;
    onexn_status st = onexn_pack_device_workspace_size(C_out, N, &need);
    if (st != ONEXN_OK) return st;
    if (!workspace || workspace_bytes < need)
        return fail(ONEXN_EINVAL, "pack_device: needs %zu bytes of workspace, got %zu", need, workspace_bytes);
    const int G = C_out / N, K = KH * KW * C_in;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    unsigned int *cnt = static_cast<unsigned int *>(workspace);
    pack_count_kernel<<<G, kThreads, 0, s>>>(mask, K, cnt);
    pack_p_kernel<<<1, kThreads, 0, s>>>(cnt, G, P);
    if (wdtype == ONEXN_BF16)
        pack_fill_kernel<true><<<G, kThreads, 0, s>>>(W, mask, C_in, KH, KW, N, P, I, D, t_cap);
    else
        pack_fill_kernel<false><<<G, kThreads, 0, s>>>(W, mask, C_in, KH, KW, N, P, I, D, t_cap);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "pack_device: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}
