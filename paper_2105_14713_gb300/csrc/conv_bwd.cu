// Backward passes of the 1xN-pruned convolution with the mask held fixed
// (fine-tuning the pruned network, Sec. 4.1): the input gradient and the
// gradient of the kept weights, in BSR order.
//
// Input gradient dx = the transposed masked convolution of dy.  For a
// stride-1 layer it is itself a convolution: dy (padded by d(K-1) - p)
// with the flipped, transposed weights Wt[c][(T-1-tap)*C_out + o] =
// W[o][tap*C_in + c] (T = KH*KW taps), so it runs on the forward tcgen05
// GEMM: decode (P, I, D) into W, transpose it per tap with the tap order
// reversed, and launch the GEMM on (dy, Wt).  A strided layer runs the same
// convolution on dy scattered onto a zero grid dilated by the stride.
// Padding beyond d(K-1) uses a direct kernel over the decoded W.
//
// Kept-weight gradient dW[o][k] = sum_p dy[p][o] * xcol[p][k] (k = tap*C_in
// + c, xcol the im2col view of x): a GEMM with the pixels as its long
// reduction dimension, run as dW^T[k][o] (M = K rows, N = C_out columns) so
// that the large operand, xcol, is the A operand: it is transposed once into
// pixel-contiguous rows (pixels padded to 64 with zeros) and, for fp32, split
// into tf32 high and low parts on the fly by the GEMM's split warps; dy is
// the small B operand, transposed with its tf32 split (fp32) and per-32-pixel
// column sums for the bias gradient.  The GEMM runs in split mode (items of
// pixel slices, one accumulator slot each) and a gather kernel adds each kept
// block's S slots in slice order into dD[z][n] = dW[g*N + n][I[z]] (fp32),
// only for the kept blocks.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "onexn_internal.h"

#include <cuda_bf16.h>

using onexn::ConvArgs;
using onexn::fail;

namespace {

constexpr int kTile = 32;           // weight transpose tiles: 32 x 32 elements, 32 x 8 threads
constexpr int kPixPad = 64;         // pixels padded to the bf16 K chunk

__device__ __forceinline__ float tf32_rna(float v)
{
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;\n" : "=r"(r) : "f"(v));
    return __uint_as_float(r);
}

template <typename T>
__device__ __forceinline__ float to_f(T v)
{
    if constexpr (sizeof(T) == 4) return v;
    else return __bfloat162float(v);
}

// Pixel-contiguous copies of the two operands of the weight-gradient GEMM
// (both K-major in the pixel index p, pixels padded to P_pad with zeros).
// One launch, two roles:
//   dy role   dYt[o][p] = dY[p][o] (fp32: as its tf32 rounding `hi` and the
//             rest `lo`), and the sums of each 32-pixel block, colsum[o][p/32]
//             (the bias gradient's first stage);
//   xcol role XcolT[tap*C + c][p] = x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c]
//             (0 outside the image).
// A CTA moves 64-pixel x 64-channel tiles through shared memory: 16-byte
// loads along channels, 16-byte stores along pixels.  bf16 tiles pair two
// pixels of one channel in a 32-bit shared word.  Each warp covers a slab of
// the tile whose rows fall on distinct banks on both sides (fp32: 8 channel
// quads x 4 pixels in, 4 channels x 8 pixel quads out; bf16: 4 channel
// octets x 8 pixel pairs in, 4 channels x 8 pixel octets out).  xcol CTAs
// are numbered tap-fastest, so the taps of one pixel range run back to back
// and re-read their x rows from L2.
constexpr int kXT = 64;                          // pixels and channels per tile
constexpr int kXcolTiles = 4;                    // pixel tiles per xcol CTA
constexpr int kColBlock = 32;                    // pixels per column-sum block

struct TransposeGrid {
    int n_dy;                                    // dy CTAs (one 64-pixel tile each)
    int cb_dy;                                   // 64-channel blocks of dy
    int cb_x;                                    // 64-channel blocks of x
    int taps;
    int n_x;                                     // xcol CTAs
};

__device__ __forceinline__ uint32_t bf16_pair(uint32_t a, uint32_t b, int hi)
{
    // (a.half[hi], b.half[hi]) as (low, high) halves of one word
    return __byte_perm(a, b, hi ? 0x7632 : 0x5410);
}

template <typename T>
__global__ void __launch_bounds__(256)
wgrad_transpose_kernel(const ConvArgs a, const T *__restrict__ dy, int P_pad, const TransposeGrid g,
                       const onexn::FastDiv div_hw, const onexn::FastDiv div_wo, T *__restrict__ xcol,
                       T *__restrict__ hi, T *__restrict__ lo, float *__restrict__ colsum, int n_pb)
{
    constexpr bool kF32 = sizeof(T) == 4;
    __shared__ uint32_t tile[kXT * (kXT + 1)];   // fp32: [64 ch][65]; bf16: [64 ch][33] pixel pairs
    __shared__ int src[kXcolTiles * kXT];        // source row of each pixel, or -1
    constexpr int kLd = kF32 ? kXT + 1 : kXT / 2 + 1;
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    const bool dy_role = static_cast<int>(blockIdx.x) < g.n_dy;
    int c0, tap = 0, pb, n_tiles, Cn;
    const T *base;
    if (dy_role) {
        const int b = blockIdx.x;
        c0 = (b % g.cb_dy) * kXT;
        pb = (b / g.cb_dy) * kXT;
        n_tiles = 1;
        Cn = a.C_out;
        base = dy;
        for (int i = tid; i < kXT; i += 256) src[i] = pb + i < a.P_pix ? pb + i : -1;
    } else {
        const int b = blockIdx.x - g.n_dy;
        tap = b % g.taps;
        const int rest = b / g.taps;
        c0 = (rest % g.cb_x) * kXT;
        pb = (rest / g.cb_x) * (kXcolTiles * kXT);
        n_tiles = min(kXcolTiles, (P_pad - pb) / kXT);
        Cn = a.C;
        base = static_cast<const T *>(a.x);
        const int kh = tap / a.KW, kw = tap - (tap / a.KW) * a.KW;
        const int hw = a.Ho * a.Wo;
        for (int i = tid; i < kXcolTiles * kXT; i += 256) {
            const int p = pb + i;
            int sp = -1;
            if (p < a.P_pix) {
                const uint32_t bb = div_hw.div(static_cast<uint32_t>(p));
                const uint32_t r = static_cast<uint32_t>(p) - bb * hw;
                const int oh = static_cast<int>(div_wo.div(r)), ow = static_cast<int>(r) - oh * a.Wo;
                const int ih = oh * a.sh - a.ph + kh * a.dh, iw = ow * a.sw - a.pw + kw * a.dw;
                if (ih >= 0 && ih < a.H && iw >= 0 && iw < a.W) sp = (static_cast<int>(bb) * a.H + ih) * a.W + iw;
            }
            src[i] = sp;
        }
    }
    __syncthreads();
    for (int tt = 0; tt < n_tiles; ++tt) {
        const int p0 = pb + tt * kXT;
        const int *s = src + tt * kXT;
        if constexpr (kF32) {
            // in: channel quad q, pixels i + 16k
            const int q = (lane & 7) + 8 * (w & 1), i = (lane >> 3) + 4 * (w >> 1);
            const bool c_ok = c0 + 4 * q < Cn;
            float4 v[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int sp = s[i + 16 * k];
                v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (sp >= 0 && c_ok)
                    v[k] = __ldg(reinterpret_cast<const float4 *>(base + static_cast<int64_t>(sp) * Cn + c0 + 4 * q));
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                uint32_t *t = tile + (4 * q) * kLd + i + 16 * k;
                t[0] = __float_as_uint(v[k].x);
                t[kLd] = __float_as_uint(v[k].y);
                t[2 * kLd] = __float_as_uint(v[k].z);
                t[3 * kLd] = __float_as_uint(v[k].w);
            }
        } else {
            // in: channel octet q, pixels 2r and 2r + 1
            const int q = (lane & 3) + 4 * (w & 1), r = (lane >> 2) + 8 * (w >> 1);
            const bool c_ok = c0 + 8 * q < Cn;
            const int s0 = s[2 * r], s1 = s[2 * r + 1];
            uint4 u0 = make_uint4(0u, 0u, 0u, 0u), u1 = u0;
            if (s0 >= 0 && c_ok)
                u0 = __ldg(reinterpret_cast<const uint4 *>(base + static_cast<int64_t>(s0) * Cn + c0 + 8 * q));
            if (s1 >= 0 && c_ok)
                u1 = __ldg(reinterpret_cast<const uint4 *>(base + static_cast<int64_t>(s1) * Cn + c0 + 8 * q));
            const uint32_t x0[4] = {u0.x, u0.y, u0.z, u0.w}, x1[4] = {u1.x, u1.y, u1.z, u1.w};
            uint32_t *t = tile + (8 * q) * kLd + r;
#pragma unroll
            for (int j = 0; j < 8; ++j) t[j * kLd] = bf16_pair(x0[j >> 1], x1[j >> 1], j & 1);
        }
        __syncthreads();
        if constexpr (kF32) {
            // out: channel rows c + 16k, pixel quad q
            const int q = (lane & 7) + 8 * (w & 1), c = (lane >> 3) + 4 * (w >> 1);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int row = c + 16 * k;
                const uint32_t *t = tile + row * kLd + 4 * q;
                const float4 v = make_float4(__uint_as_float(t[0]), __uint_as_float(t[1]), __uint_as_float(t[2]),
                                             __uint_as_float(t[3]));
                const bool ok = c0 + row < Cn;
                if (dy_role) {
                    float cs = (v.x + v.y) + (v.z + v.w);
                    cs += __shfl_xor_sync(0xffffffffu, cs, 1);
                    cs += __shfl_xor_sync(0xffffffffu, cs, 2);
                    cs += __shfl_xor_sync(0xffffffffu, cs, 4);
                    if (!ok) continue;
                    const int64_t o = static_cast<int64_t>(c0 + row);
                    if ((lane & 7) == 0) colsum[o * n_pb + p0 / kColBlock + (w & 1)] = cs;
                    const float4 h = make_float4(tf32_rna(v.x), tf32_rna(v.y), tf32_rna(v.z), tf32_rna(v.w));
                    const float4 l = make_float4(v.x - h.x, v.y - h.y, v.z - h.z, v.w - h.w);
                    *reinterpret_cast<float4 *>(hi + o * P_pad + p0 + 4 * q) = h;
                    *reinterpret_cast<float4 *>(lo + o * P_pad + p0 + 4 * q) = l;
                } else if (ok) {
                    const int64_t k_row = static_cast<int64_t>(tap) * Cn + c0 + row;
                    *reinterpret_cast<float4 *>(xcol + k_row * P_pad + p0 + 4 * q) = v;
                }
            }
        } else {
            // out: channel rows c + 32k, pixel octet q (pixel pairs 4q .. 4q + 3)
            const int q = lane & 7, c = (lane >> 3) + 4 * w;
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const int row = c + 32 * k;
                const uint32_t *t = tile + row * kLd + 4 * q;
                const uint4 v = make_uint4(t[0], t[1], t[2], t[3]);
                const bool ok = c0 + row < Cn;
                if (dy_role) {
                    float cs = 0.f;
                    const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int m = 0; m < 4; ++m)
                        cs += __uint_as_float(u[m] << 16) + __uint_as_float(u[m] & 0xffff0000u);
                    cs += __shfl_xor_sync(0xffffffffu, cs, 1);
                    cs += __shfl_xor_sync(0xffffffffu, cs, 2);
                    if (!ok) continue;
                    const int64_t o = static_cast<int64_t>(c0 + row);
                    if ((lane & 3) == 0) colsum[o * n_pb + p0 / kColBlock + (q >> 2)] = cs;
                    *reinterpret_cast<uint4 *>(hi + o * P_pad + p0 + 8 * q) = v;
                } else if (ok) {
                    const int64_t k_row = static_cast<int64_t>(tap) * Cn + c0 + row;
                    *reinterpret_cast<uint4 *>(xcol + k_row * P_pad + p0 + 8 * q) = v;
                }
            }
        }
        __syncthreads();
    }
}

// db[o] = sum of colsum[o][0 .. n_pb), one warp per channel, fixed order.
__global__ void __launch_bounds__(256)
bias_grad_kernel(const float *__restrict__ colsum, int n_pb, int C_out, float *__restrict__ db)
{
    const int o = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (o >= C_out) return;
    const float *row = colsum + static_cast<int64_t>(o) * n_pb;
    float s = 0.f;
    for (int i = lane; i < n_pb; i += 32) s += row[i];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) db[o] = s;
}

// dD[z][n] = sum over the S slices of the GEMM partial at row I[z] (the
// GEMM computes dW^T: rows k, columns o) and column g*N + n, for every kept
// block z of col-group g (found by binary search in P).  Partial slot
// i = slice * tiles + tile holds [BN/4][128] float4 (column quad, row).
__global__ void __launch_bounds__(256)
wgrad_gather_kernel(const float *__restrict__ partials, const int32_t *__restrict__ P, const int32_t *__restrict__ I,
                    int G, int N, int64_t t, int bn, int tiles, int n_tn, int S, float *__restrict__ dD)
{
    const int64_t slot_f = static_cast<int64_t>(128) * bn;
    for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < t * N;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t z = e / N;
        const int n = static_cast<int>(e - z * N);
        int lo = 0, hi = G;                       // the g with P[g] <= z < P[g + 1]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(P + mid) <= z) lo = mid; else hi = mid;
        }
        const int o = lo * N + n, k = __ldg(I + z);
        const int tile = (k / 128) * n_tn + o / bn;
        const int col = o % bn, row = k % 128;
        const int64_t off = (static_cast<int64_t>(col / 4) * 128 + row) * 4 + (col & 3);
        float s = 0.f;
        for (int sl = 0; sl < S; ++sl) s += __ldg(partials + (static_cast<int64_t>(sl) * tiles + tile) * slot_f + off);
        dD[e] = s;
    }
}

__global__ void zero_f32_kernel(float *p, int64_t n)
{
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        p[i] = 0.f;
}

// Wt[c][(T-1-tap)*C_out + o] = W[o][tap*C_in + c] (and the lo part for fp32).
template <typename T>
__global__ void __launch_bounds__(kTile * 8)
flip_transpose_kernel(const T *__restrict__ W, const T *__restrict__ W_lo, int C_out, int C_in, int taps,
                      T *__restrict__ Wt, T *__restrict__ Wt_lo)
{
    __shared__ T tile[2][kTile][kTile + 1];
    const int c0 = blockIdx.x * kTile, o0 = blockIdx.y * kTile, tap = blockIdx.z;
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int64_t K = static_cast<int64_t>(taps) * C_in, Kt = static_cast<int64_t>(taps) * C_out;
    constexpr bool kLo = sizeof(T) == 4;
    for (int i = ty; i < kTile; i += 8) {
        const int o = o0 + i, c = c0 + tx;
        const bool in = o < C_out && c < C_in;
        const int64_t at = static_cast<int64_t>(o) * K + static_cast<int64_t>(tap) * C_in + c;
        tile[0][i][tx] = in ? W[at] : T(0.f);
        if (kLo) tile[1][i][tx] = in ? W_lo[at] : T(0.f);
    }
    __syncthreads();
    const int ftap = taps - 1 - tap;
    for (int i = ty; i < kTile; i += 8) {
        const int c = c0 + i, o = o0 + tx;
        if (c >= C_in || o >= C_out) continue;
        const int64_t at = static_cast<int64_t>(c) * Kt + static_cast<int64_t>(ftap) * C_out + o;
        Wt[at] = tile[0][tx][i];
        if (kLo) Wt_lo[at] = tile[1][tx][i];
    }
}

// Direct input gradient (any stride): one thread per 16-byte channel vector
// of one input pixel; for every tap that maps it onto an output pixel, the
// dot product over the output channels with the decoded W (fp32: hi + lo,
// which is the weight exactly).
template <typename T>
__global__ void __launch_bounds__(256)
dgrad_direct_kernel(const ConvArgs a, const T *__restrict__ W, const T *__restrict__ W_lo, const T *__restrict__ dy,
                    T *__restrict__ dx, int accumulate)
{
    constexpr int kV = 16 / sizeof(T);
    const int n_vec = a.C / kV;
    const int64_t total = static_cast<int64_t>(a.B) * a.H * a.W * n_vec;
    const int64_t K = static_cast<int64_t>(a.KH) * a.KW * a.C;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int cv = static_cast<int>(i % n_vec);
        const int64_t q = i / n_vec;
        const int iw = static_cast<int>(q % a.W);
        const int ih = static_cast<int>((q / a.W) % a.H);
        const int64_t b = q / (static_cast<int64_t>(a.W) * a.H);
        const int c0 = cv * kV;
        float acc[kV];
#pragma unroll
        for (int j = 0; j < kV; ++j) acc[j] = 0.f;
        for (int kh = 0; kh < a.KH; ++kh) {
            const int th = ih + a.ph - kh * a.dh;
            if (th < 0 || th % a.sh) continue;
            const int oh = th / a.sh;
            if (oh >= a.Ho) continue;
            for (int kw = 0; kw < a.KW; ++kw) {
                const int tw = iw + a.pw - kw * a.dw;
                if (tw < 0 || tw % a.sw) continue;
                const int ow = tw / a.sw;
                if (ow >= a.Wo) continue;
                const T *dyr = dy + ((b * a.Ho + oh) * a.Wo + ow) * a.C_out;
                const int64_t kcol = static_cast<int64_t>(kh * a.KW + kw) * a.C + c0;
                for (int o = 0; o < a.C_out; ++o) {
                    const float d = to_f(dyr[o]);
                    const T *wr = W + o * K + kcol;
#pragma unroll
                    for (int j = 0; j < kV; ++j) {
                        float w = to_f(wr[j]);
                        if constexpr (sizeof(T) == 4) w += W_lo[o * K + kcol + j];
                        acc[j] = fmaf(w, d, acc[j]);
                    }
                }
            }
        }
        T *out = dx + q * a.C + c0;
#pragma unroll
        for (int j = 0; j < kV; ++j) {
            const float v = accumulate ? acc[j] + to_f(out[j]) : acc[j];
            if constexpr (sizeof(T) == 4) out[j] = v;
            else out[j] = __float2bfloat16_rn(v);
        }
    }
}

bool aligned(const void *p, uintptr_t n) { return (reinterpret_cast<uintptr_t>(p) & (n - 1)) == 0; }
size_t round256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

int grid_cap(int64_t work, int per_block, int sms)
{
    const int64_t b = (work + per_block - 1) / per_block;
    const int64_t cap = static_cast<int64_t>(sms) * 16;
    return static_cast<int>(b < 1 ? 1 : b < cap ? b : cap);
}

// The transposed convolution that computes dx, or false if the forward
// kernel cannot run it (then the direct kernel does).  For stride 1 it reads
// dy itself; for stride s it reads dy scattered onto a zero grid dilated by
// s (dy[oh] at row oh*s; Hd = (Ho-1)*s + 1 + r rows, r = the rows of x past
// the last window), so that the same stride-1 convolution with the flipped
// weights gives dx (s*s more multiply-adds, on the tensor cores).
bool dgrad_as_conv(const ConvArgs &a, int dtype, ConvArgs *t)
{
    const int ph = a.dh * (a.KH - 1) - a.ph, pw = a.dw * (a.KW - 1) - a.pw;
    if (ph < 0 || pw < 0) return false;
    const int rh = (a.H + 2 * a.ph - a.dh * (a.KH - 1) - 1) % a.sh;
    const int rw = (a.W + 2 * a.pw - a.dw * (a.KW - 1) - 1) % a.sw;
    const int Hd = (a.Ho - 1) * a.sh + 1 + rh, Wd = (a.Wo - 1) * a.sw + 1 + rw;
    ConvArgs c{};
    c.B = a.B; c.H = Hd; c.W = Wd; c.C = a.C_out; c.C_out = a.C;
    c.KH = a.KH; c.KW = a.KW; c.sh = 1; c.sw = 1; c.ph = ph; c.pw = pw; c.dh = a.dh; c.dw = a.dw;
    c.Ho = a.H; c.Wo = a.W; c.P_pix = a.B * a.H * a.W;
    c.N = 1; c.t = 0;
    // the transposed convolution's output is x's grid exactly
    if (Hd + 2 * ph - a.dh * (a.KH - 1) != a.H || Wd + 2 * pw - a.dw * (a.KW - 1) != a.W) return false;
    if (static_cast<int64_t>(a.B) * Hd * Wd >= (int64_t(1) << 31)) return false;
    if (!onexn::tc_supports(c, dtype)) return false;
    *t = c;
    return true;
}

struct DgradWs {
    size_t w, wt, dyd, total;
};

DgradWs dgrad_ws(const ConvArgs &a, int dtype)
{
    DgradWs l{};
    const size_t wb = onexn::tc_weights_bytes(a, dtype);
    l.w = 0;
    l.wt = wb;
    l.dyd = 2 * wb;
    l.total = 2 * wb;
    ConvArgs tr{};
    if ((a.sh > 1 || a.sw > 1) && dgrad_as_conv(a, dtype, &tr))
        l.total += round256(static_cast<size_t>(tr.B) * tr.H * tr.W * tr.C * (dtype == ONEXN_F32 ? 4 : 2));
    return l;
}

// dyd[b][i][j][:] = dy[b][i/sh][j/sw][:] where sh | i and sw | j (inside dy),
// else 0; one thread per 16-byte channel vector.
template <typename T>
__global__ void __launch_bounds__(256)
dilate_kernel(const T *__restrict__ dy, int B, int Ho, int Wo, int C, int sh, int sw, int Hd, int Wd,
              T *__restrict__ dyd)
{
    constexpr int kV = 16 / sizeof(T);
    const int n_vec = C / kV;
    const int64_t total = static_cast<int64_t>(B) * Hd * Wd * n_vec;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int cv = static_cast<int>(i % n_vec);
        const int64_t q = i / n_vec;
        const int j = static_cast<int>(q % Wd), r = static_cast<int>((q / Wd) % Hd);
        const int64_t b = q / (static_cast<int64_t>(Wd) * Hd);
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r % sh == 0 && j % sw == 0 && r / sh < Ho && j / sw < Wo)
            v = __ldg(reinterpret_cast<const uint4 *>(dy + ((b * Ho + r / sh) * Wo + j / sw) * C) + cv);
        reinterpret_cast<uint4 *>(dyd + q * C)[cv] = v;
    }
}

struct WgradWs {
    int64_t P_pad;
    int n_pb;
    onexn::TcSplitPlan plan;
    size_t xcol, dy_hi, dy_lo, colsum, part, total;
};

WgradWs wgrad_ws(const ConvArgs &a, int dtype)
{
    WgradWs l{};
    const size_t es = dtype == ONEXN_F32 ? 4 : 2;
    const int64_t K = static_cast<int64_t>(a.KH) * a.KW * a.C;
    l.P_pad = (static_cast<int64_t>(a.P_pix) + kPixPad - 1) / kPixPad * kPixPad;
    l.n_pb = static_cast<int>(l.P_pad / kColBlock);
    l.plan = onexn::tc_split_plan(static_cast<int>(K), a.C_out, l.P_pad, dtype);
    l.xcol = 0;
    l.dy_hi = round256(static_cast<size_t>(K) * l.P_pad * es);
    l.dy_lo = l.dy_hi + round256(static_cast<size_t>(a.C_out) * l.P_pad * es);
    l.colsum = l.dy_lo + (dtype == ONEXN_F32 ? round256(static_cast<size_t>(a.C_out) * l.P_pad * es) : 0);
    l.part = l.colsum + round256(static_cast<size_t>(a.C_out) * l.n_pb * 4);
    l.total = l.part + round256(l.plan.partial_bytes);
    return l;
}

onexn_status bwd_shape(const onexn_conv_desc *desc, int N, int64_t t, int dtype, ConvArgs *a, const char *who)
{
    onexn_status st = onexn::detail::check_shape(desc, N, t, dtype, 0, a);
    if (st != ONEXN_OK) return st;
    if (a->C_out % 8) return fail(ONEXN_EUNSUPPORTED, "%s: C_out=%d must be a multiple of 8", who, a->C_out);
    if (a->C_out / a->N > 65535) return fail(ONEXN_EUNSUPPORTED, "%s: more than 65535 col-groups", who);
    return ONEXN_OK;
}

}  // namespace

extern "C" onexn_status onexn_conv_bwd_data_workspace_size(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                                                           size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "conv_bwd_data: bytes is NULL");
    ConvArgs a{};
    onexn_status st = bwd_shape(desc, N, t, dtype, &a, "conv_bwd_data");
    if (st != ONEXN_OK) return st;
    *bytes = dgrad_ws(a, dtype).total;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_bwd_data(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I,
                                            const void *D, int N, int64_t t, const void *dy, void *dx, int dtype,
                                            unsigned flags, void *workspace, size_t workspace_bytes, void *stream)
{
    onexn::clear_error();
    ConvArgs a{};
    onexn_status st = bwd_shape(desc, N, t, dtype, &a, "conv_bwd_data");
    if (st != ONEXN_OK) return st;
    if (flags & ~ONEXN_ACCUMULATE) return fail(ONEXN_EINVAL, "conv_bwd_data: unknown flags");
    const size_t es = dtype == ONEXN_F32 ? 4 : 2;
    const size_t x_bytes = static_cast<size_t>(a.B) * a.H * a.W * a.C * es;
    const size_t y_bytes = static_cast<size_t>(a.P_pix) * a.C_out * es;
    if (x_bytes == 0) return ONEXN_OK;
    if (!dy || !dx || !P || (t > 0 && (!I || !D))) return fail(ONEXN_EINVAL, "conv_bwd_data: NULL pointer");
    if (!aligned(dy, 16) || !aligned(dx, 16)) return fail(ONEXN_EINVAL, "conv_bwd_data: dy and dx must be 16-byte aligned");
    {
        const uintptr_t d0 = reinterpret_cast<uintptr_t>(dy), x0 = reinterpret_cast<uintptr_t>(dx);
        if (d0 < x0 + x_bytes && x0 < d0 + y_bytes) return fail(ONEXN_EINVAL, "conv_bwd_data: dy and dx overlap");
    }
    const DgradWs L = dgrad_ws(a, dtype);
    if (!workspace || workspace_bytes < L.total)
        return fail(ONEXN_EINVAL, "conv_bwd_data: needs %zu bytes of workspace, got %zu", L.total, workspace_bytes);
    if (!aligned(workspace, 256)) return fail(ONEXN_EINVAL, "conv_bwd_data: workspace must be 256-byte aligned");
    a.P = P; a.I = I; a.D = D; a.x = nullptr; a.y = nullptr;
    cudaError_t e = onexn::device_status_ptr(&a.status);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: status word: %s", cudaGetErrorString(e));
    int sms = 0;
    e = onexn::device_sm_count(&sms);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: %s", cudaGetErrorString(e));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    const size_t n_w = static_cast<size_t>(a.C_out) * a.KH * a.KW * a.C;
    // the masked dense weights (fp32: hi, then lo), as the forward decodes them
    e = onexn::tc_decode(a, dtype, ws + L.w, onexn::tc_weights_bytes(a, dtype), s);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: decode: %s", cudaGetErrorString(e));
    const bool acc = (flags & ONEXN_ACCUMULATE) != 0;
    ConvArgs tr{};
    if (dgrad_as_conv(a, dtype, &tr)) {
        const dim3 grid((a.C + kTile - 1) / kTile, (a.C_out + kTile - 1) / kTile, a.KH * a.KW);
        const dim3 block(kTile, 8);
        void *wt = ws + L.wt;
        if (dtype == ONEXN_F32) {
            const float *w = reinterpret_cast<const float *>(ws + L.w);
            float *t_hi = static_cast<float *>(wt);
            flip_transpose_kernel<float><<<grid, block, 0, s>>>(w, w + n_w, a.C_out, a.C, a.KH * a.KW, t_hi,
                                                                 t_hi + n_w);
        } else {
            const __nv_bfloat16 *w = reinterpret_cast<const __nv_bfloat16 *>(ws + L.w);
            flip_transpose_kernel<__nv_bfloat16><<<grid, block, 0, s>>>(w, nullptr, a.C_out, a.C, a.KH * a.KW,
                                                                         static_cast<__nv_bfloat16 *>(wt), nullptr);
        }
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: transpose: %s", cudaGetErrorString(e));
        const void *src = dy;
        if (a.sh > 1 || a.sw > 1) {
            void *dyd = ws + L.dyd;
            const int kv = dtype == ONEXN_F32 ? 4 : 8;
            const int g = grid_cap(static_cast<int64_t>(tr.B) * tr.H * tr.W * (tr.C / kv), 256, sms);
            if (dtype == ONEXN_F32)
                dilate_kernel<float><<<g, 256, 0, s>>>(static_cast<const float *>(dy), a.B, a.Ho, a.Wo, a.C_out, a.sh,
                                                        a.sw, tr.H, tr.W, static_cast<float *>(dyd));
            else
                dilate_kernel<__nv_bfloat16><<<g, 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(dy), a.B, a.Ho, a.Wo,
                                                                a.C_out, a.sh, a.sw, tr.H, tr.W,
                                                                static_cast<__nv_bfloat16 *>(dyd));
            e = cudaGetLastError();
            if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: dilate: %s", cudaGetErrorString(e));
            src = dyd;
        }
        tr.x = src; tr.y = dx; tr.residual = acc ? dx : nullptr; tr.bias = nullptr; tr.relu = 0;
        tr.status = a.status;
        const void *wt_lo = dtype == ONEXN_F32 ? static_cast<const void *>(static_cast<float *>(wt) + n_w) : nullptr;
        e = onexn::tc_gemm_weights(tr, dtype, wt, wt_lo, nullptr, s);
        if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: GEMM: %s", cudaGetErrorString(e));
        return ONEXN_OK;
    }
    const int kv = dtype == ONEXN_F32 ? 4 : 8;
    const int grid = grid_cap(static_cast<int64_t>(a.B) * a.H * a.W * (a.C / kv), 256, sms);
    if (dtype == ONEXN_F32) {
        const float *w = reinterpret_cast<const float *>(ws + L.w);
        dgrad_direct_kernel<float><<<grid, 256, 0, s>>>(a, w, w + n_w, static_cast<const float *>(dy),
                                                         static_cast<float *>(dx), acc ? 1 : 0);
    } else {
        const __nv_bfloat16 *w = reinterpret_cast<const __nv_bfloat16 *>(ws + L.w);
        dgrad_direct_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(a, w, nullptr, static_cast<const __nv_bfloat16 *>(dy),
                                                                 static_cast<__nv_bfloat16 *>(dx), acc ? 1 : 0);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_data: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_bwd_weight_workspace_size(const onexn_conv_desc *desc, int N, int dtype,
                                                             size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "conv_bwd_weight: bytes is NULL");
    ConvArgs a{};
    onexn_status st = bwd_shape(desc, N, 0, dtype, &a, "conv_bwd_weight");
    if (st != ONEXN_OK) return st;
    *bytes = wgrad_ws(a, dtype).total;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_bwd_weight(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I, int N,
                                              int64_t t, const void *x, const void *dy, float *dD, float *db,
                                              int dtype, void *workspace, size_t workspace_bytes, void *stream)
{
    onexn::clear_error();
    ConvArgs a{};
    onexn_status st = bwd_shape(desc, N, t, dtype, &a, "conv_bwd_weight");
    if (st != ONEXN_OK) return st;
    if (!P || (t > 0 && (!I || !dD))) return fail(ONEXN_EINVAL, "conv_bwd_weight: NULL pointer");
    if (a.P_pix > 0 && (!x || !dy)) return fail(ONEXN_EINVAL, "conv_bwd_weight: x or dy is NULL");
    if (!aligned(x, 16) || !aligned(dy, 16) || !aligned(dD, 4) || !aligned(db, 4))
        return fail(ONEXN_EINVAL, "conv_bwd_weight: x and dy must be 16-byte aligned, dD and db 4-byte aligned");
    const WgradWs L = wgrad_ws(a, dtype);
    if (!workspace || workspace_bytes < L.total)
        return fail(ONEXN_EINVAL, "conv_bwd_weight: needs %zu bytes of workspace, got %zu", L.total, workspace_bytes);
    if (!aligned(workspace, 256)) return fail(ONEXN_EINVAL, "conv_bwd_weight: workspace must be 256-byte aligned");
    int sms = 0;
    cudaError_t e = onexn::device_sm_count(&sms);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_weight: %s", cudaGetErrorString(e));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (a.P_pix == 0) {
        // no pixels: every gradient is zero
        if (t > 0) zero_f32_kernel<<<grid_cap(t * N, 256, sms), 256, 0, s>>>(dD, t * N);
        if (db) zero_f32_kernel<<<grid_cap(a.C_out, 256, sms), 256, 0, s>>>(db, a.C_out);
        e = cudaGetLastError();
        return e == cudaSuccess ? ONEXN_OK : fail(ONEXN_ECUDA, "conv_bwd_weight: %s", cudaGetErrorString(e));
    }
    a.x = x;
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    const int K = a.KH * a.KW * a.C;
    if (L.P_pad > INT32_MAX / 2) return fail(ONEXN_EINVAL, "conv_bwd_weight: too many pixels");
    const int P_pad = static_cast<int>(L.P_pad);
    TransposeGrid tg{};
    tg.cb_dy = (a.C_out + kXT - 1) / kXT;
    tg.cb_x = (a.C + kXT - 1) / kXT;
    tg.taps = a.KH * a.KW;
    const int64_t n_dy = static_cast<int64_t>(P_pad / kXT) * tg.cb_dy;
    const int64_t n_x = static_cast<int64_t>((P_pad / kXT + kXcolTiles - 1) / kXcolTiles) * tg.cb_x * tg.taps;
    if (n_dy + n_x > INT32_MAX) return fail(ONEXN_EINVAL, "conv_bwd_weight: too many pixels x channels");
    tg.n_dy = static_cast<int>(n_dy);
    tg.n_x = static_cast<int>(n_x);
    const unsigned n_cta = static_cast<unsigned>(n_dy + n_x);
    const onexn::FastDiv div_hw(static_cast<uint32_t>(a.Ho * a.Wo)), div_wo(static_cast<uint32_t>(a.Wo));
    float *colsum = reinterpret_cast<float *>(ws + L.colsum);
    if (dtype == ONEXN_F32) {
        wgrad_transpose_kernel<float><<<n_cta, 256, 0, s>>>(
            a, static_cast<const float *>(dy), P_pad, tg, div_hw, div_wo, reinterpret_cast<float *>(ws + L.xcol),
            reinterpret_cast<float *>(ws + L.dy_hi), reinterpret_cast<float *>(ws + L.dy_lo), colsum, L.n_pb);
    } else {
        wgrad_transpose_kernel<__nv_bfloat16><<<n_cta, 256, 0, s>>>(
            a, static_cast<const __nv_bfloat16 *>(dy), P_pad, tg, div_hw, div_wo,
            reinterpret_cast<__nv_bfloat16 *>(ws + L.xcol), reinterpret_cast<__nv_bfloat16 *>(ws + L.dy_hi), nullptr,
            colsum, L.n_pb);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_weight: transpose: %s", cudaGetErrorString(e));
    // the GEMM dW^T[K][C_out] = XcolT[K][P_pad] . dYt[C_out][P_pad]^T, in pixel slices
    ConvArgs g{};
    g.B = 1; g.H = 1; g.W = K; g.C = P_pad; g.C_out = a.C_out;
    g.KH = 1; g.KW = 1; g.sh = 1; g.sw = 1; g.ph = 0; g.pw = 0; g.dh = 1; g.dw = 1;
    g.Ho = 1; g.Wo = K; g.P_pix = K; g.N = 1; g.t = 0;
    g.x = ws + L.xcol; g.y = ws + L.xcol;
    e = onexn::device_status_ptr(&g.status);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_weight: status word: %s", cudaGetErrorString(e));
    float *part = reinterpret_cast<float *>(ws + L.part);
    e = onexn::tc_gemm_split(g, dtype, ws + L.dy_hi, dtype == ONEXN_F32 ? ws + L.dy_lo : nullptr, part, L.plan, s);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_weight: GEMM: %s", cudaGetErrorString(e));
    if (t > 0)
        wgrad_gather_kernel<<<grid_cap(t * a.N, 256, sms), 256, 0, s>>>(part, P, I, a.C_out / a.N, a.N, t, L.plan.bn,
                                                                        L.plan.tiles, L.plan.n_tn, L.plan.split_s, dD);
    if (db) bias_grad_kernel<<<(a.C_out + 7) / 8, 256, 0, s>>>(colsum, L.n_pb, a.C_out, db);
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_bwd_weight: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}
