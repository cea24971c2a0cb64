// CUDA-core (FFMA) kernel of the 1xN-pruned convolution, Eq. 7:
//   Y[p, gN:(g+1)N] = sum_{z=P[g]}^{P[g+1]-1} X[p, I[z]] * D[z, :]
//
// One CTA owns a tile of MT = 128 consecutive output pixels and a tile of
// output columns.  Columns are processed in "slices" of NS <= 32 columns
// (NS divides N; a slice lies inside one col-group, so every slice of group
// g walks the same kept list I[P[g]..P[g+1]) with its own D columns).
//
// The index space k = (kh*KW + kw)*C + c is walked in chunks of one tap and
// KC = 32 channels.  For each chunk the CTA stages the im2col slab
// X[p, k0 .. k0+KC) of its 128 pixels into shared memory, transposed to
// [channel][pixel] so that a warp reads one kept index for 4 pixels per lane
// with one conflict-free 16-byte load.  Because every group's kept list is
// sorted, each slice consumes its entries chunk by chunk with a pointer that
// only moves forward.  Each thread accumulates 4 pixels x NS columns x SPW
// slices in fp32 registers; weights D[z, co:co+NS) are warp-uniform loads.
// The next chunk is loaded into registers while the current one is computed
// (register double buffering) and stored after it, one barrier per chunk.
#include "conv_common.cuh"
#include "onexn_internal.h"

namespace onexn {

namespace {

constexpr int kThreads = 128;  // 4 warps
constexpr int kMT = 128;       // output pixels per CTA
constexpr int kR = 4;          // pixels per thread (one float4 of the staged row)
constexpr int kKC = 32;        // channels per chunk
constexpr int kXS = kMT + 4;   // staged row stride (floats): 16-B aligned, 4 mod 32 banks

template <typename TIN>
struct Stage;

// fp32 input: a pixel's 32 channels are 8 16-byte vectors.  A warp stages 32
// pixels; lane l takes pixel (l % 16) of a 16-pixel half and vectors
// 2i + l/16, so a warp load covers 16 full 32-byte sectors and the transposed
// stores hit 32 distinct banks.
template <>
struct Stage<float> {
    static constexpr int kPix = 2;                    // pixels staged per thread
    static constexpr int kIter = 4;                   // vectors per pixel per thread
    using V = float4;
    __device__ static int pixel(int warp, int lane, int j) { return 32 * warp + 16 * j + (lane & 15); }
    __device__ static int vec(int lane, int i) { return 2 * i + (lane >> 4); }
    __device__ static void store(float (*xs)[kXS], int p, int v, const V &a)
    {
        xs[4 * v + 0][p] = a.x; xs[4 * v + 1][p] = a.y;
        xs[4 * v + 2][p] = a.z; xs[4 * v + 3][p] = a.w;
    }
};

// bf16 input: a pixel's 32 channels are 4 16-byte vectors of 8.  Lane l takes
// pixel 32*warp + l and vector i, so the 8 transposed stores per vector hit
// 32 distinct banks.  Values are widened to fp32 when staged.
template <>
struct Stage<__nv_bfloat16> {
    static constexpr int kPix = 1;
    static constexpr int kIter = 4;
    using V = uint4;
    __device__ static int pixel(int warp, int lane, int) { return 32 * warp + lane; }
    __device__ static int vec(int, int i) { return i; }
    __device__ static void store(float (*xs)[kXS], int p, int v, const V &a)
    {
        xs[8 * v + 0][p] = bf16lo(a.x); xs[8 * v + 1][p] = bf16hi(a.x);
        xs[8 * v + 2][p] = bf16lo(a.y); xs[8 * v + 3][p] = bf16hi(a.y);
        xs[8 * v + 4][p] = bf16lo(a.z); xs[8 * v + 5][p] = bf16hi(a.z);
        xs[8 * v + 6][p] = bf16lo(a.w); xs[8 * v + 7][p] = bf16hi(a.w);
    }
};

template <typename TIN, int NS, int SPW>
__global__ void __launch_bounds__(kThreads)
fma_conv_kernel(const ConvArgs a)
{
    // Entries examined per step of the kept-list walk (bounded by registers).
    constexpr int kBatch = NS >= 32 ? 2 : 4;
    using S = Stage<TIN>;
    using V = typename S::V;
    constexpr int kElemPerVec = 16 / sizeof(TIN);
    __shared__ __align__(16) float xs[2][kKC][kXS];

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int pix0 = blockIdx.x * kMT;
    const int n_slices = a.C_out / NS;
    const int slice0 = (blockIdx.y * (kThreads / 32) + warp) * SPW;
    const TIN *__restrict__ x = static_cast<const TIN *>(a.x);
    const TIN *__restrict__ Dw = static_cast<const TIN *>(a.D);

    // ---- staging role: the input position of this thread's staged pixels ----
    int sb[S::kPix], sih[S::kPix], siw[S::kPix];
#pragma unroll
    for (int j = 0; j < S::kPix; ++j) {
        const int p = pix0 + S::pixel(warp, lane, j);
        if (p < a.P_pix) {
            const int hw = a.Ho * a.Wo;
            const int b = p / hw, r = p - b * hw;
            const int oh = r / a.Wo, ow = r - oh * a.Wo;
            sb[j] = b; sih[j] = oh * a.sh - a.ph; siw[j] = ow * a.sw - a.pw;
        } else {
            sb[j] = -1; sih[j] = 0; siw[j] = 0;
        }
    }

    const int n_cchunk = (a.C + kKC - 1) / kKC;
    const int n_chunks = a.KH * a.KW * n_cchunk;
    V stage[S::kPix][S::kIter];

    auto load_chunk = [&](int chunk) {
        const int tap = chunk / n_cchunk;
        const int c0 = (chunk - tap * n_cchunk) * kKC;
        const int kh = tap / a.KW, kw = tap - kh * a.KW;
#pragma unroll
        for (int j = 0; j < S::kPix; ++j) {
            const int ih = sih[j] + kh * a.dh, iw = siw[j] + kw * a.dw;
            const bool ok = sb[j] >= 0 && ih >= 0 && ih < a.H && iw >= 0 && iw < a.W;
            const TIN *row = x + ((static_cast<int64_t>(ok ? sb[j] : 0) * a.H + (ok ? ih : 0)) * a.W +
                                  (ok ? iw : 0)) * a.C + c0;
#pragma unroll
            for (int i = 0; i < S::kIter; ++i) {
                const int v = S::vec(lane, i);
                const bool in = ok && (c0 + v * kElemPerVec < a.C);
                stage[j][i] = in ? __ldg(reinterpret_cast<const V *>(row) + v) : V{};
            }
        }
    };
    auto store_chunk = [&](int buf) {
#pragma unroll
        for (int j = 0; j < S::kPix; ++j)
#pragma unroll
            for (int i = 0; i < S::kIter; ++i)
                S::store(xs[buf], S::pixel(warp, lane, j), S::vec(lane, i), stage[j][i]);
    };

    // ---- compute role: kept-list pointers of this warp's slices ----
    int zptr[SPW], zend[SPW], dcol[SPW];
#pragma unroll
    for (int s = 0; s < SPW; ++s) {
        const int sl = slice0 + s;
        if (sl < n_slices) {
            const int col = sl * NS, g = col / a.N;
            zptr[s] = clampi(__ldg(a.P + g), 0, a.t);
            zend[s] = clampi(__ldg(a.P + g + 1), zptr[s], a.t);
            dcol[s] = col - g * a.N;
        } else {
            zptr[s] = zend[s] = 0; dcol[s] = 0;
        }
    }

    float acc[SPW][kR][NS];
#pragma unroll
    for (int s = 0; s < SPW; ++s)
#pragma unroll
        for (int r = 0; r < kR; ++r)
#pragma unroll
            for (int n = 0; n < NS; ++n) acc[s][r][n] = 0.f;

    load_chunk(0);
    store_chunk(0);
    __syncthreads();

    for (int chunk = 0; chunk < n_chunks; ++chunk) {
        const int buf = chunk & 1;
        if (chunk + 1 < n_chunks) load_chunk(chunk + 1);

        const int tap = chunk / n_cchunk;
        const int k0 = tap * a.C + (chunk - tap * n_cchunk) * kKC;
        const int kend = k0 + min(kKC, a.C - (chunk - tap * n_cchunk) * kKC);
        const float *xrow = &xs[buf][0][4 * lane];

#pragma unroll
        for (int s = 0; s < SPW; ++s) {
            int z = zptr[s];
            const int ze = zend[s];
            while (z < ze) {
                int kk[kBatch];
#pragma unroll
                for (int j = 0; j < kBatch; ++j)
                    kk[j] = (z + j < ze) ? __ldg(a.I + z + j) : 0x7fffffff;
                float4 xv[kBatch];
                float d[kBatch][NS];
#pragma unroll
                for (int j = 0; j < kBatch; ++j) {
                    const int cl = clampi(kk[j] - k0, 0, kKC - 1);
                    xv[j] = *reinterpret_cast<const float4 *>(xrow + cl * kXS);
                    load_row<NS>(Dw + static_cast<int64_t>(min(z + j, ze - 1)) * a.N + dcol[s], d[j]);
                }
                int n_ok = 0;
#pragma unroll
                for (int j = 0; j < kBatch; ++j) n_ok += (kk[j] < kend) ? 1 : 0;
#pragma unroll
                for (int j = 0; j < kBatch; ++j) {
                    if (j < n_ok) {
#pragma unroll
                        for (int n = 0; n < NS; ++n) {
                            acc[s][0][n] = fmaf(xv[j].x, d[j][n], acc[s][0][n]);
                            acc[s][1][n] = fmaf(xv[j].y, d[j][n], acc[s][1][n]);
                            acc[s][2][n] = fmaf(xv[j].z, d[j][n], acc[s][2][n]);
                            acc[s][3][n] = fmaf(xv[j].w, d[j][n], acc[s][3][n]);
                        }
                    }
                }
                z += n_ok;
                if (n_ok < kBatch) break;
            }
            zptr[s] = z;
        }

        if (chunk + 1 < n_chunks) store_chunk(buf ^ 1);
        __syncthreads();
    }

    // ---- epilogue: bias, ReLU, NHWC store ----
    TIN *__restrict__ y = static_cast<TIN *>(a.y);
    const bool vec_ok = (a.C_out % (16 / sizeof(TIN))) == 0;
#pragma unroll
    for (int s = 0; s < SPW; ++s) {
        const int sl = slice0 + s;
        if (sl >= n_slices) continue;
        const int col = sl * NS;
        float bv[NS];
#pragma unroll
        for (int n = 0; n < NS; ++n) bv[n] = a.bias ? __ldg(a.bias + col + n) : 0.f;
#pragma unroll
        for (int r = 0; r < kR; ++r) {
            const int p = pix0 + 4 * lane + r;
            if (p >= a.P_pix) continue;
            float v[NS];
#pragma unroll
            for (int n = 0; n < NS; ++n) {
                v[n] = acc[s][r][n] + bv[n];
                if (a.relu) v[n] = fmaxf(v[n], 0.f);
            }
            store_row<NS>(y + static_cast<int64_t>(p) * a.C_out + col, v, vec_ok);
        }
    }
}

// Columns per warp ~16 (NS * SPW), so every instantiation holds 64 fp32
// accumulators per thread, except NS = 32 (128).
template <int NS> struct SlicesPerWarp { static constexpr int v = NS >= 16 ? 1 : 16 / NS; };

template <typename TIN, int NS>
cudaError_t launch_ns(const ConvArgs &a, cudaStream_t st)
{
    constexpr int SPW = SlicesPerWarp<NS>::v;
    const int n_slices = a.C_out / NS;
    const int cols_per_cta = (kThreads / 32) * SPW;            // slices per CTA
    dim3 grid((a.P_pix + kMT - 1) / kMT, (n_slices + cols_per_cta - 1) / cols_per_cta);
    fma_conv_kernel<TIN, NS, SPW><<<grid, kThreads, 0, st>>>(a);
    return cudaGetLastError();
}

template <typename TIN>
cudaError_t launch_t(const ConvArgs &a, cudaStream_t st)
{
    // Widest slice that divides N.
    if (a.N % 32 == 0) return launch_ns<TIN, 32>(a, st);
    if (a.N % 16 == 0) return launch_ns<TIN, 16>(a, st);
    if (a.N % 8 == 0) return launch_ns<TIN, 8>(a, st);
    if (a.N % 4 == 0) return launch_ns<TIN, 4>(a, st);
    if (a.N % 2 == 0) return launch_ns<TIN, 2>(a, st);
    return launch_ns<TIN, 1>(a, st);
}

}  // namespace

cudaError_t launch_fma(const ConvArgs &a, int dtype, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    if (dtype == ONEXN_F32) return launch_t<float>(a, st);
    return launch_t<__nv_bfloat16>(a, st);
}

}  // namespace onexn
