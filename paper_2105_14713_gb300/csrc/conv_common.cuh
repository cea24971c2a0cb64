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
    int relu;               // activation after bias (+ residual): 0 none, 1 ReLU, 2 ReLU6
    const void *residual;   // nullable, NHWC like y: y = act(acc + bias + residual)
    unsigned int *status;   // library status word (device): bits set by kernels on failure
    // Fused depthwise producer of the A operand (fp32 tensor-core GEMM of a
    // 1x1 layer only; x is then unused): A[p][c] = relu6(dw_b[c] +
    // sum_{kh,kw} dw_w[kh*3+kw][c] * dw_x[b, oh*dw_s - 1 + kh, ow*dw_s - 1 + kw, c])
    // for output pixel p = (b, oh, ow), zero padding.
    const float *dw_x;      // nullable: NHWC [B][dw_H][dw_W][C]
    const float *dw_w;      // [9][C], tap-major
    const float *dw_b;      // [C] or nullptr
    int dw_H, dw_W, dw_s;
};

// Bits of the device status word (read by onexn_device_status).
constexpr unsigned int kStatusTimeout = 1u;
constexpr unsigned int kStatusBadInput = 2u;   // the validation kernel found a malformed (P, I)

// Host: SM count of the current device (cached per device).
cudaError_t device_sm_count(int *sms);
// Host: the same, or 152 (GB300) if it cannot be queried; for cost models
// and tile planning, which only need an estimate.
int device_sms_or_default();
// Host: device address of the status word of the current device.
cudaError_t device_status_ptr(unsigned int **p);

__device__ __forceinline__ int clampi(int v, int lo, int hi) { return min(max(v, lo), hi); }

// The activation of ConvArgs::relu: 0 none, 1 max(v, 0), 2 min(max(v, 0), 6).
__device__ __forceinline__ float activate(float v, int kind)
{
    if (kind >= 1) v = fmaxf(v, 0.f);
    if (kind == 2) v = fminf(v, 6.f);
    return v;
}
// The same with the kind fixed at compile time (no branch per value).
template <int kKind>
__device__ __forceinline__ float activate_c(float v)
{
    if constexpr (kKind >= 1) v = fmaxf(v, 0.f);
    if constexpr (kKind == 2) v = fminf(v, 6.f);
    return v;
}

// Division of 32-bit unsigned integers by an invariant divisor d >= 1 with
// one multiply-high, after Granlund and Montgomery, "Division by invariant
// integers using multiplication" (PLDI 1994), Fig. 4.1:
//   l = ceil(log2 d), m = floor(2^32 (2^l - d) / d) + 1,
//   t = mulhi(m, n), q = (t + ((n - t) >> min(l, 1))) >> max(l - 1, 0).
// The constants are computed on the host; exact for every 32-bit n.
struct FastDiv {
    uint32_t d = 1, m = 1, s1 = 0, s2 = 0;
    FastDiv() = default;
    __host__ explicit FastDiv(uint32_t dd) : d(dd)
    {
        uint32_t l = 0;
        while (l < 32 && (uint64_t(1) << l) < dd) ++l;
        m = static_cast<uint32_t>(((uint64_t(1) << 32) * ((uint64_t(1) << l) - dd)) / dd + 1);
        s1 = l < 1 ? l : 1;
        s2 = l > 1 ? l - 1 : 0;
    }
    __device__ __forceinline__ uint32_t div(uint32_t n) const
    {
        const uint32_t t = __umulhi(m, n);
        return (t + ((n - t) >> s1)) >> s2;
    }
};

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---- cp.async (16 bytes, L2 only; src_bytes = 0 zero-fills the destination) ----
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// ---- mbarriers (CTA scope) ----
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}\n" ::"r"(bar)
                 : "memory");
}
// One bounded try: the warp is suspended until the phase completes or about
// 0.1 ms pass (suspend-time hint), so waiting warps do not take issue slots.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(100000u)
        : "memory");
    return ok != 0;
}
// Wait for the phase with the given parity to complete, for at most ~2^31
// SM cycles (about one second).  Returns false on expiry.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > (1ll << 31)) return false;
    }
    return true;
}

// Single test of a phase, without suspending.
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait (~2^31 SM cycles) that sleeps `ns` nanoseconds between tests,
// for warps that are not on the critical path: they stay off the issue slots.
__device__ __forceinline__ bool mbar_wait_backoff(uint32_t bar, uint32_t parity, unsigned ns)
{
    if (mbar_test(bar, parity)) return true;
    const long long t0 = clock64();
    do {
        __nanosleep(ns);
        if (mbar_test(bar, parity)) return true;
    } while (clock64() - t0 <= (1ll << 31));
    return false;
}

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
