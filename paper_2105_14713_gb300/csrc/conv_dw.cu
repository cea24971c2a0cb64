// onexn_dwconv_fwd: the dense depthwise convolution of MobileNet-V2's
// inverted-residual block (the KHxKW per-channel convolution between the
// pruned expand and project 1x1 convolutions; it is not pruned):
//   y[b,oh,ow,c] = act(bias[c] + sum_{kh,kw} W[c][kh][kw]
//                  * x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c])
// with zero padding.  One thread computes one 16-byte vector of channels
// (4 fp32 / 8 bf16) of one output pixel: consecutive threads take
// consecutive channel vectors of a pixel, so every x load and y store of a
// warp is contiguous.  It streams x and y once (plus the halo re-reads from
// L2) and is bound by HBM bandwidth.
#include "conv_common.cuh"
#include "onexn_internal.h"

using onexn::fail;

namespace {

template <typename T>
struct DwVec;
template <>
struct DwVec<float> {
    static constexpr int kV = 4;
    static __device__ __forceinline__ void load(const float *p, float (&v)[4])
    {
        const float4 q = __ldg(reinterpret_cast<const float4 *>(p));
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
    }
    static __device__ __forceinline__ void store(float *p, const float (&v)[4])
    {
        *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    }
};
template <>
struct DwVec<__nv_bfloat16> {
    static constexpr int kV = 8;
    static __device__ __forceinline__ void load(const __nv_bfloat16 *p, float (&v)[8])
    {
        const uint4 q = __ldg(reinterpret_cast<const uint4 *>(p));
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            v[2 * i] = onexn::bf16lo(w[i]);
            v[2 * i + 1] = onexn::bf16hi(w[i]);
        }
    }
    static __device__ __forceinline__ void store(__nv_bfloat16 *p, const float (&v)[8])
    {
        *reinterpret_cast<uint4 *>(p) =
            make_uint4(onexn::pack_bf16x2(v[0], v[1]), onexn::pack_bf16x2(v[2], v[3]),
                       onexn::pack_bf16x2(v[4], v[5]), onexn::pack_bf16x2(v[6], v[7]));
    }
};

// Raw 16-byte vector of kV channels; converted to fp32 at use.
template <typename T>
struct DwRaw;
template <>
struct DwRaw<float> {
    float4 q;
    __device__ __forceinline__ void load(const float *p) { q = __ldg(reinterpret_cast<const float4 *>(p)); }
    __device__ __forceinline__ void zero() { q = make_float4(0.f, 0.f, 0.f, 0.f); }
    __device__ __forceinline__ float operator[](int j) const
    {
        return j == 0 ? q.x : j == 1 ? q.y : j == 2 ? q.z : q.w;
    }
};
template <>
struct DwRaw<__nv_bfloat16> {
    uint4 q;
    __device__ __forceinline__ void load(const __nv_bfloat16 *p) { q = __ldg(reinterpret_cast<const uint4 *>(p)); }
    __device__ __forceinline__ void zero() { q = make_uint4(0u, 0u, 0u, 0u); }
    __device__ __forceinline__ float operator[](int j) const
    {
        const uint32_t w = (j >> 1) == 0 ? q.x : (j >> 1) == 1 ? q.y : (j >> 1) == 2 ? q.z : q.w;
        return (j & 1) ? onexn::bf16hi(w) : onexn::bf16lo(w);
    }
};

// KS = 3: the 3x3 form of MobileNet-V2, fully unrolled: the thread's
// kV x 9 weights (contiguous in W[C][3][3]) come in as float4 loads and all
// nine input vectors are requested before the first multiply, so one
// memory latency covers a pixel.  KS = 0: any KH x KW, tap by tap.
// Launched as a programmatic dependent: the wait comes before the first
// read of x, and the next kernel may launch once every thread is done.
template <typename T, int KS>
__global__ void __launch_bounds__(256)
dw_conv_kernel(const onexn::ConvArgs a, const float *__restrict__ W, const onexn::FastDiv div_vec,
               const onexn::FastDiv div_hw, const onexn::FastDiv div_wo)
{
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    using V = DwVec<T>;
    constexpr int kV = V::kV;
    const uint32_t n_vec = static_cast<uint32_t>(a.C / kV);
    const uint32_t total = static_cast<uint32_t>(a.P_pix) * n_vec;
    const uint32_t hw = static_cast<uint32_t>(a.Ho * a.Wo);
    const T *x = static_cast<const T *>(a.x);
    T *y = static_cast<T *>(a.y);
    for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
        const uint32_t p = div_vec.div(i);
        const int c0 = static_cast<int>(i - p * n_vec) * kV;
        const uint32_t b = div_hw.div(p);
        const uint32_t r = p - b * hw;
        const int oh = static_cast<int>(div_wo.div(r));
        const int ow = static_cast<int>(r) - oh * a.Wo;
        const T *xb = x + static_cast<int64_t>(b) * a.H * a.W * a.C + c0;
        float acc[kV];
#pragma unroll
        for (int j = 0; j < kV; ++j) acc[j] = a.bias ? __ldg(a.bias + c0 + j) : 0.f;
        if constexpr (KS > 0) {
            constexpr int kT = KS * KS;
            float w[kV * kT];
            const float4 *wp = reinterpret_cast<const float4 *>(W + static_cast<int64_t>(c0) * kT);
#pragma unroll
            for (int q = 0; q < kV * kT / 4; ++q) {
                const float4 v = __ldg(wp + q);
                w[4 * q] = v.x; w[4 * q + 1] = v.y; w[4 * q + 2] = v.z; w[4 * q + 3] = v.w;
            }
            DwRaw<T> v[kT];
#pragma unroll
            for (int kh = 0; kh < KS; ++kh) {
                const int ih = oh * a.sh - a.ph + kh * a.dh;
#pragma unroll
                for (int kw = 0; kw < KS; ++kw) {
                    const int iw = ow * a.sw - a.pw + kw * a.dw;
                    if (ih >= 0 && ih < a.H && iw >= 0 && iw < a.W)
                        v[kh * KS + kw].load(xb + (static_cast<int64_t>(ih) * a.W + iw) * a.C);
                    else
                        v[kh * KS + kw].zero();
                }
            }
#pragma unroll
            for (int t = 0; t < kT; ++t)
#pragma unroll
                for (int j = 0; j < kV; ++j) acc[j] = fmaf(w[j * kT + t], v[t][j], acc[j]);
        } else {
            const int taps = a.KH * a.KW;
            for (int kh = 0; kh < a.KH; ++kh) {
                const int ih = oh * a.sh - a.ph + kh * a.dh;
                if (ih < 0 || ih >= a.H) continue;
                for (int kw = 0; kw < a.KW; ++kw) {
                    const int iw = ow * a.sw - a.pw + kw * a.dw;
                    if (iw < 0 || iw >= a.W) continue;
                    float v[kV];
                    V::load(xb + (static_cast<int64_t>(ih) * a.W + iw) * a.C, v);
                    const int tap = kh * a.KW + kw;
#pragma unroll
                    for (int j = 0; j < kV; ++j)
                        acc[j] = fmaf(__ldg(W + static_cast<int64_t>(c0 + j) * taps + tap), v[j], acc[j]);
                }
            }
        }
#pragma unroll
        for (int j = 0; j < kV; ++j) acc[j] = onexn::activate(acc[j], a.relu);
        V::store(y + static_cast<int64_t>(p) * a.C + c0, acc);
    }
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

bool aligned(const void *p, uintptr_t n) { return (reinterpret_cast<uintptr_t>(p) & (n - 1)) == 0; }

}  // namespace

extern "C" onexn_status onexn_dwconv_fwd(const onexn_conv_desc *desc, const float *W, const float *bias,
                                         const void *x, void *y, int dtype, unsigned flags, void *stream)
{
    onexn::clear_error();
    if (!desc) return fail(ONEXN_EINVAL, "dwconv: desc is NULL");
    int Ho = 0, Wo = 0;
    onexn_status st = onexn_conv_out_shape(desc, &Ho, &Wo);
    if (st != ONEXN_OK) return st;
    if (dtype != ONEXN_F32 && dtype != ONEXN_BF16) return fail(ONEXN_EINVAL, "dwconv: unknown dtype %d", dtype);
    if (desc->C_in != desc->C_out)
        return fail(ONEXN_EINVAL, "dwconv: C_in=%d and C_out=%d differ", desc->C_in, desc->C_out);
    const int v = dtype == ONEXN_F32 ? 4 : 8;
    if (desc->C_in % v) return fail(ONEXN_EINVAL, "dwconv: C=%d must be a multiple of %d", desc->C_in, v);
    if (flags & ~(ONEXN_RELU | ONEXN_RELU6)) return fail(ONEXN_EINVAL, "dwconv: unknown flags");
    const int64_t npix = static_cast<int64_t>(desc->B) * Ho * Wo;
    if (npix * (desc->C_in / v) >= (int64_t(1) << 31) || npix >= (int64_t(1) << 31))
        return fail(ONEXN_EINVAL, "dwconv: too large (2^31 channel vectors at most)");
    if (npix > 0 && (!x || !y || !W)) return fail(ONEXN_EINVAL, "dwconv: x, y or W is NULL");
    if (!aligned(x, 16) || !aligned(y, 16) || !aligned(W, 16) || !aligned(bias, 4))
        return fail(ONEXN_EINVAL, "dwconv: x, y and W must be 16-byte aligned, bias 4-byte aligned");
    if (npix > 0) {
        const size_t es = dtype == ONEXN_F32 ? 4 : 2;
        const uintptr_t x0 = reinterpret_cast<uintptr_t>(x),
                        x1 = x0 + static_cast<size_t>(desc->B) * desc->H * desc->W * desc->C_in * es;
        const uintptr_t y0 = reinterpret_cast<uintptr_t>(y), y1 = y0 + static_cast<size_t>(npix) * desc->C_in * es;
        if (x0 < y1 && y0 < x1) return fail(ONEXN_EINVAL, "dwconv: x and y overlap");
    } else {
        return ONEXN_OK;
    }
    onexn::ConvArgs a{};
    a.x = x; a.y = y; a.bias = bias;
    a.B = desc->B; a.H = desc->H; a.W = desc->W; a.C = desc->C_in; a.C_out = desc->C_out;
    a.KH = desc->KH; a.KW = desc->KW;
    a.sh = desc->stride_h; a.sw = desc->stride_w; a.ph = desc->pad_h; a.pw = desc->pad_w;
    a.dh = desc->dil_h; a.dw = desc->dil_w; a.Ho = Ho; a.Wo = Wo;
    a.P_pix = static_cast<int>(npix);
    a.relu = (flags & ONEXN_RELU6) ? 2 : (flags & ONEXN_RELU) ? 1 : 0;
    int sms = 0;
    cudaError_t e = onexn::device_sm_count(&sms);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "dwconv: %s", cudaGetErrorString(e));
    const int64_t work = npix * (desc->C_in / v);
    const int64_t blocks = (work + 255) / 256;
    const int grid = static_cast<int>(blocks < static_cast<int64_t>(sms) * 16 ? blocks : static_cast<int64_t>(sms) * 16);
    const onexn::FastDiv div_vec(static_cast<uint32_t>(desc->C_in / v)), div_hw(static_cast<uint32_t>(Ho * Wo)),
        div_wo(static_cast<uint32_t>(Wo));
    const bool k3 = desc->KH == 3 && desc->KW == 3;
    void (*kern)(const onexn::ConvArgs, const float *, const onexn::FastDiv, const onexn::FastDiv,
                 const onexn::FastDiv);
    if (dtype == ONEXN_F32)
        kern = k3 ? dw_conv_kernel<float, 3> : dw_conv_kernel<float, 0>;
    else
        kern = k3 ? dw_conv_kernel<__nv_bfloat16, 3> : dw_conv_kernel<__nv_bfloat16, 0>;
    // a programmatic dependent of the previous kernel on the stream: its
    // launch overlaps that kernel's tail; the kernel waits before reading
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(256);
    cfg.stream = static_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, a, W, div_vec, div_hw, div_wo);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "dwconv: launch failed: %s", cudaGetErrorString(e));
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "dwconv: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}
