// CUDA-core (FFMA) kernel of the 1xN-pruned convolution, Eq. 7:
//   Y[p, gN:(g+1)N] = sum_{z=P[g]}^{P[g+1]-1} X[p, I[z]] * D[z, :]
//
// Work units.  A unit is MT = 256 consecutive output pixels x 64 output
// columns.  Columns are handled in slices of NS <= 8 (NS divides N; a slice
// lies inside one col-group, so every slice of group g walks the same kept
// list I[P[g] .. P[g+1]) with its own D columns).  The kernel is persistent:
// one CTA per SM walks units blockIdx.x, blockIdx.x + gridDim.x, ...
//
// Warp roles (12 warps):
//  * 8 consumer warps.  Consumer w owns SPW slices (8 columns) of the unit
//    and all 256 pixels: lane l accumulates pixels 4l..4l+3 and
//    128+4l..128+4l+3 in fp32 registers (64 accumulators).
//  * 4 producer warps.  Producer w copies and transposes pixels
//    64w .. 64w+63 of every chunk.
//
// The index space k = (kh*KW + kw)*C + c is walked in chunks of one tap and
// KC = 32 channels; the kept lists are sorted, so every slice consumes its
// entries chunk by chunk.  Per chunk:
//   producers: cp.async copies the im2col slab X[p, k0 .. k0+KC) (zero in the
//     padding) into a landing buffer one chunk ahead, then transpose it into
//     a [channel][pixel] fp32 stage of a 4-deep ring and arrive on the
//     stage's "full" mbarrier;
//   consumers: the next <= 32 kept entries of each slice were loaded one
//     chunk earlier with one coalesced load each (lane j holds I[z+j] and
//     D[z+j, co:co+NS)).  Wait "full", count the entries inside the chunk
//     with a ballot, park their weights in a per-warp shared buffer (fp32),
//     start the loads for the next chunk, and for each kept block broadcast
//     its channel with a shuffle, read 8 pixels with two 16-byte shared
//     loads and its NS weights with broadcast shared loads, and issue 8*NS
//     FFMAs; then arrive on the stage's "empty" mbarrier.
// Consumers only wait for data, never for each other, so a slice with more
// kept blocks in one chunk does not stall the others.  Every mbarrier wait
// is bounded (~1 s); on expiry the kernel records ONEXN_ETIMEOUT in the
// library status word and returns.
#include "conv_common.cuh"
#include "onexn_internal.h"

namespace onexn {

namespace {

constexpr int kConsumers = 8;
constexpr int kProducers = 4;
constexpr int kThreads = 32 * (kConsumers + kProducers);
constexpr int kMT = 256;            // output pixels per unit
constexpr int kColsPerUnit = 64;    // 8 consumer warps x 8 columns
constexpr int kKC = 32;             // channels per chunk
constexpr int kXS = kMT + 4;        // transposed row stride (floats): 16-B aligned, = 4 mod 32
constexpr int kStages = 4;          // transposed stages in the ring
constexpr int kLand = 2;            // landing buffers per producer (copies in flight: kLand-1)

template <typename TIN>
struct Tile {
    static constexpr int kElemPerVec = 16 / sizeof(TIN);          // 4 (fp32) or 8 (bf16)
    static constexpr int kVecPerPix = kKC / kElemPerVec;          // 8 or 4
    static constexpr int kLandBytes = kMT * kKC * sizeof(TIN);    // one landing buffer
    static constexpr int kXsBytes = kKC * kXS * 4;
    static constexpr int kDsBytes = kConsumers * 32 * 8 * 4;        // per warp: [32 rows][8 cols] fp32
    static constexpr int kDsOff = kLand * kLandBytes + kStages * kXsBytes;
    static constexpr int kBarOff = kDsOff + kDsBytes;
    static constexpr int kSmem = kBarOff + 2 * kStages * 8;
};

// 16-byte vector v of pixel p sits at vector slot land_swz(p, v) of the
// pixel's landing row (XOR swizzle).  128-bit shared accesses are serviced
// a quarter-warp (8 lanes) at a time; with the lane mappings of the copy and
// transposition below every quarter-warp touches 8 distinct 16-byte bank
// groups (fp32; bf16 rows are 64 B and stay within 2-way).
template <typename TIN>
__device__ __forceinline__ int land_swz(int p, int v)
{
    if constexpr (sizeof(TIN) == 4) return v ^ (2 * ((p >> 2) & 3));   // 8 vectors per 128-B row
    else return v ^ ((p >> 1) & 3);                                     // 4 vectors per 64-B row
}

// Copy role: the pixel (within the producer's 64) that lane l copies in step i.
// fp32: lane pairs take one pixel (two adjacent vectors = one 32-B sector);
// a quarter-warp takes pixels k, k+4, k+8, k+12 so that their swizzles differ.
template <typename TIN>
__device__ __forceinline__ int copy_pixel(int lane, int i)
{
    const int m = lane >> 1;
    if constexpr (sizeof(TIN) == 4) return 16 * i + (m >> 2) + 4 * (m & 3);
    else return 16 * i + m;
}

__device__ __forceinline__ float4 lds128(uint32_t a)
{
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];\n"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(a)
                 : "memory");
    return v;
}
__device__ __forceinline__ float lds32(uint32_t a)
{
    float v;
    asm volatile("ld.shared.f32 %0, [%1];\n" : "=f"(v) : "r"(a) : "memory");
    return v;
}

template <typename TIN, int NS, int SPW>
__global__ void __launch_bounds__(kThreads, 1)
fma_conv_kernel(const ConvArgs a, const int n_units, const int n_ct)
{
    using T = Tile<TIN>;
    extern __shared__ __align__(128) unsigned char smem[];
    TIN *land = reinterpret_cast<TIN *>(smem);                                   // [kLand][MT][KC]
    float *xs_all = reinterpret_cast<float *>(smem + kLand * T::kLandBytes);     // [kStages][KC][XS]
    const uint32_t bar_full = smem_u32(smem + T::kBarOff);                       // [kStages]
    const uint32_t bar_empty = bar_full + 8 * kStages;                           // [kStages]

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(bar_full + 8 * s, kProducers);
            mbar_init(bar_empty + 8 * s, kConsumers);
        }
        fence_mbar_init();
    }
    __syncthreads();

    const int n_cchunk = (a.C + kKC - 1) / kKC;
    const int n_chunks = a.KH * a.KW * n_cchunk;
    const int my_units = blockIdx.x < n_units ? (n_units - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    const int n_items = my_units * n_chunks;

    if (warp >= kConsumers) {
        // ======================= producers =======================
        const int pw = warp - kConsumers;
        const TIN *__restrict__ x = static_cast<const TIN *>(a.x);
        const int q = lane & 1;
        // pixels of this lane in the copy role: 64pw + copy_pixel(lane, i), i < 4
        int cb[4], cih[4], ciw[4];
        int cur_unit = -1;
        auto set_unit = [&](int u) {
            const int pt = u / n_ct;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int p = pt * kMT + 64 * pw + copy_pixel<TIN>(lane, i);
                if (p < a.P_pix) {
                    const int hw = a.Ho * a.Wo;
                    const int b = p / hw, r = p - b * hw;
                    const int oh = r / a.Wo, ow = r - oh * a.Wo;
                    cb[i] = b; cih[i] = oh * a.sh - a.ph; ciw[i] = ow * a.sw - a.pw;
                } else {
                    cb[i] = -1; cih[i] = 0; ciw[i] = 0;
                }
            }
        };
        auto issue = [&](int item) {
            if (item < n_items) {
                const int ui = item / n_chunks, chunk = item - ui * n_chunks;
                const int u = blockIdx.x + ui * gridDim.x;
                if (u != cur_unit) { set_unit(u); cur_unit = u; }
                const int tap = chunk / n_cchunk;
                const int c0 = (chunk - tap * n_cchunk) * kKC;
                const int kh = tap / a.KW, kw = tap - kh * a.KW;
                TIN *L = land + (item % kLand) * kMT * kKC;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int ih = cih[i] + kh * a.dh, iw = ciw[i] + kw * a.dw;
                    const bool ok = cb[i] >= 0 && ih >= 0 && ih < a.H && iw >= 0 && iw < a.W;
                    const TIN *row = x + ((static_cast<int64_t>(ok ? cb[i] : 0) * a.H + (ok ? ih : 0)) * a.W +
                                          (ok ? iw : 0)) * a.C + c0;
                    const int pl = 64 * pw + copy_pixel<TIN>(lane, i);
                    TIN *dst = L + pl * kKC;
#pragma unroll
                    for (int j = 0; j < T::kVecPerPix / 2; ++j) {
                        const int v = 2 * j + q;
                        const bool in = ok && (c0 + v * T::kElemPerVec < a.C);
                        cp_async16(smem_u32(dst + land_swz<TIN>(pl, v) * T::kElemPerVec),
                                   in ? row + v * T::kElemPerVec : x, in ? 16 : 0);
                    }
                }
            }
            cp_async_commit();   // always commit, so group counting stays uniform
        };

        for (int i = 0; i < kLand - 1; ++i) issue(i);
        for (int item = 0; item < n_items; ++item) {
            issue(item + kLand - 1);
            cp_async_wait<kLand - 1>();
            __syncwarp();
            const int st = item % kStages;
            if (item >= kStages && !mbar_wait(bar_empty + 8 * st, ((item / kStages) + 1) & 1)) {
                atomicOr(a.status, kStatusTimeout);
                break;
            }
            const TIN *L = land + (item % kLand) * kMT * kKC;
            float *xs = xs_all + st * kKC * kXS;
            if constexpr (sizeof(TIN) == 4) {
                const int cq = lane >> 2;                                  // channels 4cq..4cq+3
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int p = 4 * (16 * pw + (lane & 3) + 4 * i);      // pixels p..p+3
                    float4 r[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        r[e] = *reinterpret_cast<const float4 *>(L + (p + e) * kKC + 4 * land_swz<TIN>(p + e, cq));
                    *reinterpret_cast<float4 *>(xs + (4 * cq + 0) * kXS + p) = make_float4(r[0].x, r[1].x, r[2].x, r[3].x);
                    *reinterpret_cast<float4 *>(xs + (4 * cq + 1) * kXS + p) = make_float4(r[0].y, r[1].y, r[2].y, r[3].y);
                    *reinterpret_cast<float4 *>(xs + (4 * cq + 2) * kXS + p) = make_float4(r[0].z, r[1].z, r[2].z, r[3].z);
                    *reinterpret_cast<float4 *>(xs + (4 * cq + 3) * kXS + p) = make_float4(r[0].w, r[1].w, r[2].w, r[3].w);
                }
            } else {
                const int oct = lane & 3;                                  // channels 8oct..8oct+7
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const int p = 4 * (16 * pw + (lane >> 2) + 8 * i);     // pixels p..p+3
                    uint4 r[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        r[e] = *reinterpret_cast<const uint4 *>(L + (p + e) * kKC + 8 * land_swz<TIN>(p + e, oct));
                    float *o = xs + (8 * oct) * kXS + p;
#define ONEXN_T8(F, LOHI, row)                                                              \
    *reinterpret_cast<float4 *>(o + (row) * kXS) =                                          \
        make_float4(LOHI(r[0].F), LOHI(r[1].F), LOHI(r[2].F), LOHI(r[3].F));
                    ONEXN_T8(x, bf16lo, 0) ONEXN_T8(x, bf16hi, 1) ONEXN_T8(y, bf16lo, 2) ONEXN_T8(y, bf16hi, 3)
                    ONEXN_T8(z, bf16lo, 4) ONEXN_T8(z, bf16hi, 5) ONEXN_T8(w, bf16lo, 6) ONEXN_T8(w, bf16hi, 7)
#undef ONEXN_T8
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_full + 8 * st);
        }
        cp_async_wait<0>();
        return;
    }

    // ======================= consumers =======================
    const TIN *__restrict__ Dw = static_cast<const TIN *>(a.D);
    TIN *__restrict__ y = static_cast<TIN *>(a.y);
    float *ds = reinterpret_cast<float *>(smem + T::kDsOff) + warp * (32 * 8);   // [SPW][32][NS]
    const int n_slices = a.C_out / NS;
    const bool vec_ok = (a.C_out % (16 / sizeof(TIN))) == 0;
    int item = 0;
    for (int ui = 0; ui < my_units; ++ui) {
        const int u = blockIdx.x + ui * gridDim.x;
        const int pt = u / n_ct, ct = u - pt * n_ct;
        const int pix0 = pt * kMT;
        // Per slice: kept-list cursor, and the next <= 32 candidate entries
        // prefetched one chunk ahead: lane j holds I[z+j] and D[z+j, co:co+NS).
        int zptr[SPW] = {}, zend[SPW] = {}, dcol[SPW] = {}, myk[SPW];
        float myd[SPW][NS];
        auto prefetch = [&](int s) {
            const bool ok = zptr[s] + lane < zend[s];
            myk[s] = ok ? __ldg(a.I + zptr[s] + lane) : 0x7fffffff;
            if (ok) {
                load_row<NS>(Dw + static_cast<int64_t>(zptr[s] + lane) * a.N + dcol[s], myd[s]);
            } else {
#pragma unroll
                for (int n = 0; n < NS; ++n) myd[s][n] = 0.f;
            }
        };
#pragma unroll
        for (int s = 0; s < SPW; ++s) {
            const int sl = (ct * kConsumers + warp) * SPW + s;
            if (sl < n_slices) {
                const int col = sl * NS, g = col / a.N;
                zptr[s] = clampi(__ldg(a.P + g), 0, a.t);
                zend[s] = clampi(__ldg(a.P + g + 1), zptr[s], a.t);
                dcol[s] = col - g * a.N;
            } else {
                zptr[s] = zend[s] = 0; dcol[s] = 0;
            }
            prefetch(s);
        }
        float acc[SPW][8][NS];
#pragma unroll
        for (int s = 0; s < SPW; ++s)
#pragma unroll
            for (int r = 0; r < 8; ++r)
#pragma unroll
                for (int n = 0; n < NS; ++n) acc[s][r][n] = 0.f;

        int cc0 = 0, tapC = 0;                  // channel offset in the tap, tap * C
        for (int chunk = 0; chunk < n_chunks; ++chunk, ++item) {
            const int st = item % kStages;
            if (!mbar_wait(bar_full + 8 * st, (item / kStages) & 1)) {
                atomicOr(a.status, kStatusTimeout);
                return;
            }
            const int k0 = tapC + cc0;
            const int kend = k0 + min(kKC, a.C - cc0);
            cc0 += kKC;
            if (cc0 >= a.C) { cc0 = 0; tapC += a.C; }
            const uint32_t xa = smem_u32(xs_all + st * kKC * kXS + 4 * lane);
            int cnt[SPW], mycl[SPW];
            __syncwarp();                       // previous chunk's reads of ds are done
#pragma unroll
            for (int s = 0; s < SPW; ++s) {
                cnt[s] = __popc(__ballot_sync(0xffffffffu, myk[s] < kend));
                mycl[s] = clampi(myk[s] - k0, 0, kKC - 1);
                float *dst = ds + (s * 32 + lane) * NS;
                if constexpr (NS % 4 == 0) {
#pragma unroll
                    for (int n = 0; n < NS; n += 4)
                        *reinterpret_cast<float4 *>(dst + n) =
                            make_float4(myd[s][n], myd[s][n + 1], myd[s][n + 2], myd[s][n + 3]);
                } else {
#pragma unroll
                    for (int n = 0; n < NS; ++n) dst[n] = myd[s][n];
                }
                zptr[s] += cnt[s];
                prefetch(s);                    // entries of the next chunk, a chunk ahead
            }
            __syncwarp();                       // ds visible to the whole warp
#pragma unroll
            for (int s = 0; s < SPW; ++s) {
                const uint32_t dsr = smem_u32(ds + s * 32 * NS);
                const int n = cnt[s];
                if (n == 0) continue;
                // Software pipeline over two register sets (no copies): the
                // shared loads of entry j+1 are issued before the 8*NS FFMAs
                // of entry j.
                float4 xa0, xa1, xb0, xb1;
                float da[NS], db[NS];
                auto load_entry = [&](int j, float4 &v0, float4 &v1, float (&dv)[NS]) {
                    const int cl = __shfl_sync(0xffffffffu, mycl[s], j);
                    const uint32_t xad = xa + cl * (kXS * 4);
                    v0 = lds128(xad);
                    v1 = lds128(xad + 512);
                    const uint32_t dad = dsr + j * (NS * 4);
                    if constexpr (NS % 4 == 0) {
#pragma unroll
                        for (int c = 0; c < NS; c += 4) {
                            const float4 v = lds128(dad + 4 * c);
                            dv[c] = v.x; dv[c + 1] = v.y; dv[c + 2] = v.z; dv[c + 3] = v.w;
                        }
                    } else {
#pragma unroll
                        for (int c = 0; c < NS; ++c) dv[c] = lds32(dad + 4 * c);
                    }
                };
                auto fma_entry = [&](const float4 &v0, const float4 &v1, const float (&dv)[NS]) {
#pragma unroll
                    for (int c = 0; c < NS; ++c) {
                        acc[s][0][c] = fmaf(v0.x, dv[c], acc[s][0][c]);
                        acc[s][1][c] = fmaf(v0.y, dv[c], acc[s][1][c]);
                        acc[s][2][c] = fmaf(v0.z, dv[c], acc[s][2][c]);
                        acc[s][3][c] = fmaf(v0.w, dv[c], acc[s][3][c]);
                        acc[s][4][c] = fmaf(v1.x, dv[c], acc[s][4][c]);
                        acc[s][5][c] = fmaf(v1.y, dv[c], acc[s][5][c]);
                        acc[s][6][c] = fmaf(v1.z, dv[c], acc[s][6][c]);
                        acc[s][7][c] = fmaf(v1.w, dv[c], acc[s][7][c]);
                    }
                };
                load_entry(0, xa0, xa1, da);
                int j = 0;
                for (; j + 2 <= n; j += 2) {
                    load_entry(j + 1, xb0, xb1, db);
                    fma_entry(xa0, xa1, da);
                    load_entry(min(j + 2, n - 1), xa0, xa1, da);
                    fma_entry(xb0, xb1, db);
                }
                if (j < n) fma_entry(xa0, xa1, da);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_empty + 8 * st);
        }

        // ---- epilogue of the unit: bias, ReLU, NHWC store ----
#pragma unroll
        for (int s = 0; s < SPW; ++s) {
            const int sl = (ct * kConsumers + warp) * SPW + s;
            if (sl >= n_slices) continue;
            const int col = sl * NS;
            float bv[NS];
#pragma unroll
            for (int n = 0; n < NS; ++n) bv[n] = a.bias ? __ldg(a.bias + col + n) : 0.f;
#pragma unroll
            for (int r = 0; r < 8; ++r) {
                const int p = pix0 + 4 * lane + (r & 3) + 128 * (r >> 2);
                if (p >= a.P_pix) continue;
                float v[NS];
#pragma unroll
                for (int n = 0; n < NS; ++n) v[n] = acc[s][r][n] + bv[n];
                if (a.residual) {
                    float rv[NS];
                    // aligned: NS divides N, which divides C_out, and residual is 16-byte aligned
                    load_row<NS>(static_cast<const TIN *>(a.residual) + static_cast<int64_t>(p) * a.C_out + col, rv);
#pragma unroll
                    for (int n = 0; n < NS; ++n) v[n] += rv[n];
                }
#pragma unroll
                for (int n = 0; n < NS; ++n) v[n] = activate(v[n], a.relu);
                store_row<NS>(y + static_cast<int64_t>(p) * a.C_out + col, v, vec_ok);
            }
        }
    }
}

template <typename TIN, int NS>
cudaError_t launch_ns(const ConvArgs &a, cudaStream_t st)
{
    constexpr int SPW = 8 / NS;                            // 8 columns per consumer warp
    auto kern = fma_conv_kernel<TIN, NS, SPW>;
    const int smem = Tile<TIN>::kSmem;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int sms = 0;
    e = device_sm_count(&sms);
    if (e != cudaSuccess) return e;
    const int n_pt = (a.P_pix + kMT - 1) / kMT;
    const int n_ct = (a.C_out + kColsPerUnit - 1) / kColsPerUnit;
    const int n_units = n_pt * n_ct;
    const int grid = n_units < sms ? n_units : sms;
    kern<<<grid, kThreads, smem, st>>>(a, n_units, n_ct);
    return cudaGetLastError();
}

template <typename TIN>
cudaError_t launch_t(const ConvArgs &a, cudaStream_t st)
{
    // Widest slice (<= 8) that divides N; wider groups are split into slices.
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
