// Device-side helpers shared by the onexn convolution kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace onexn {

// Geometry and BSR weights of one launch (all pointers are device pointers).
struct ConvArgs {
    const void *x;          // NHWC input
    void *y;                // NHWC output
    const float *bias;      // [C_out] or nullptr
    const int32_t *P;       // [G+1]
    const int32_t *I;       // [t]
    const void *D;          // [t][N]
    int B, H, W, C;         // input
    int C_out, KH, KW;
    int sh, sw, ph, pw, dh, dw;
    int Ho, Wo;
    int N;                  // block width
    int t;                  // number of kept blocks (entries of I / rows of D)
    int P_pix;              // B * Ho * Wo
    int relu;
};

__device__ __forceinline__ int clampi(int v, int lo, int hi) { return min(max(v, lo), hi); }

// bf16 bits -> fp32 (exact).
__device__ __forceinline__ float bf16lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Load NS consecutive weights of one D row as fp32.
template <int NS>
__device__ __forceinline__ void load_row(const float *p, float (&d)[NS])
{
    if constexpr (NS % 4 == 0) {
#pragma unroll
        for (int i = 0; i < NS / 4; ++i) {
            const float4 v = __ldg(reinterpret_cast<const float4 *>(p) + i);
            d[4 * i + 0] = v.x; d[4 * i + 1] = v.y; d[4 * i + 2] = v.z; d[4 * i + 3] = v.w;
        }
    } else if constexpr (NS == 2) {
        const float2 v = __ldg(reinterpret_cast<const float2 *>(p));
        d[0] = v.x; d[1] = v.y;
    } else {
#pragma unroll
        for (int i = 0; i < NS; ++i) d[i] = __ldg(p + i);
    }
}

template <int NS>
__device__ __forceinline__ void load_row(const __nv_bfloat16 *p, float (&d)[NS])
{
    if constexpr (NS % 8 == 0) {
#pragma unroll
        for (int i = 0; i < NS / 8; ++i) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(p) + i);
            d[8 * i + 0] = bf16lo(v.x); d[8 * i + 1] = bf16hi(v.x);
            d[8 * i + 2] = bf16lo(v.y); d[8 * i + 3] = bf16hi(v.y);
            d[8 * i + 4] = bf16lo(v.z); d[8 * i + 5] = bf16hi(v.z);
            d[8 * i + 6] = bf16lo(v.w); d[8 * i + 7] = bf16hi(v.w);
        }
    } else if constexpr (NS == 4) {
        const uint2 v = __ldg(reinterpret_cast<const uint2 *>(p));
        d[0] = bf16lo(v.x); d[1] = bf16hi(v.x); d[2] = bf16lo(v.y); d[3] = bf16hi(v.y);
    } else if constexpr (NS == 2) {
        const uint32_t v = __ldg(reinterpret_cast<const unsigned int *>(p));
        d[0] = bf16lo(v); d[1] = bf16hi(v);
    } else {
        const unsigned short v = __ldg(reinterpret_cast<const unsigned short *>(p));
        d[0] = bf16lo(v);
    }
}

// Store NS consecutive fp32 results (fp32 or RNE-rounded bf16 output).
template <int NS>
__device__ __forceinline__ void store_row(float *p, const float (&v)[NS], bool vec_ok)
{
    if constexpr (NS % 4 == 0) {
        if (vec_ok) {
#pragma unroll
            for (int i = 0; i < NS / 4; ++i)
                reinterpret_cast<float4 *>(p)[i] =
                    make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
            return;
        }
    }
#pragma unroll
    for (int i = 0; i < NS; ++i) p[i] = v[i];
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

template <int NS>
__device__ __forceinline__ void store_row(__nv_bfloat16 *p, const float (&v)[NS], bool vec_ok)
{
    if constexpr (NS % 8 == 0) {
        if (vec_ok) {
#pragma unroll
            for (int i = 0; i < NS / 8; ++i)
                reinterpret_cast<uint4 *>(p)[i] =
                    make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                               pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
            return;
        }
    }
#pragma unroll
    for (int i = 0; i < NS; ++i) p[i] = __float2bfloat16_rn(v[i]);
}

}  // namespace onexn
