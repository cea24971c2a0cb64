// Measurement kernels behind the rooflines and design figures of the
// library (not part of the convolution): the fp32 FFMA rate of the GPU, and
// the issue rate of tcgen05.mma by block width N, number of issuing threads
// and A-operand source (tensor memory or shared memory).  Launch only; the
// caller times them (CUDA events) and derives the rates.
#include "conv_common.cuh"
#include "onexn_internal.h"
#include "tc_ptx.cuh"

namespace onexn {
namespace {

constexpr int kFmaChains = 8;

// Every thread runs kFmaChains independent fp32 multiply-add chains of
// `iters` steps: 2 * kFmaChains * iters flops per thread.  The sum is stored
// only if it equals a value it cannot reach, so the chains are kept.
__global__ void __launch_bounds__(256) ffma_chain_kernel(int iters, float seed, float *sink)
{
    float v[kFmaChains];
#pragma unroll
    for (int c = 0; c < kFmaChains; ++c) v[c] = seed + 0.001f * static_cast<float>(threadIdx.x + c);
    const float m = 0.999999f, a = 1e-7f;
    for (int i = 0; i < iters; ++i) {
#pragma unroll
        for (int c = 0; c < kFmaChains; ++c) v[c] = fmaf(v[c], m, a);
    }
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < kFmaChains; ++c) s += v[c];
    if (s == -12345.f) sink[blockIdx.x] = s;
}

constexpr int kProbeWarps = 8;

// Back-to-back tcgen05.mma (kind::f16, M = 128, K = 16, zero operands) issued
// by lane 0 of each of `issuers` warps into its own accumulator: 4 * iters
// MMAs per issuer.  A is read from tensor memory (kATmem) or from shared
// memory; B from shared memory.  The A source is a template parameter: a
// run-time branch between the issues slows the issue itself.  One CTA per SM (the shared-memory
// request exceeds half an SM).
template <int N, bool kATmem>
__global__ void __launch_bounds__(kProbeWarps * 32, 1) mma_issue_kernel(int iters, int issuers, unsigned int *status)
{
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    constexpr int kA = 128 * 128, kB = 256 * 128;     // 128 x 64 bf16, up to 256 x 64 bf16
    const int tid = threadIdx.x, warp = tid >> 5;
    for (int i = tid; i < (kA + kB) / 16; i += blockDim.x) reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0, 0, 0, 0);
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + kA + kB);
    const uint32_t bar = base + kA + kB + 64;         // one mbarrier per issuer
    if (tid == 0) {
        for (int w = 0; w < kProbeWarps; ++w) mbar_init(bar + 8 * w, 1);
        fence_mbar_init();
    }
    tc::fence_proxy_async_smem();
    if (warp == 0) {
        tc::tmem_alloc(smem_u32(holder), 512);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;
    if (warp < 4) {
        // A in tensor memory: columns 256..287 of every lane, zero
        uint32_t z[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) z[i] = 0u;
        tc::st_32x32b_x32(tmem + ((32u * warp) << 16) + 256, z);
        tc::st_wait();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    if (warp < issuers && (tid & 31) == 0) {
        constexpr uint32_t idesc = tc::idesc_bf16_f32(128, N);
        const uint64_t ad = tc::desc_kmajor_sw128(base), bd = tc::desc_kmajor_sw128(base + kA);
        const uint32_t d = tmem + static_cast<uint32_t>(warp) * 32;   // issuer's accumulator (N <= 32 here)
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                if constexpr (kATmem)
                    tc::mma_bf16_ta(d, tmem + 256 + 8 * kk, bd + 2 * kk, idesc, (it | kk) != 0);
                else
                    tc::mma_bf16(d, ad + 2 * kk, bd + 2 * kk, idesc, (it | kk) != 0);
            }
        }
        tc::commit(bar + 8 * warp);
        if (!mbar_wait(bar + 8 * warp, 0)) atomicOr(status, kStatusTimeout);
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 512);
    }
}

constexpr int kMmaProbeSmem = 128 * 128 + 256 * 128 + 1024 + 256 + 70000;

}  // namespace
}  // namespace onexn

using onexn::fail;

extern "C" onexn_status onexn_probe_ffma(int blocks, int iters, float *sink, void *stream)
{
    onexn::clear_error();
    if (blocks < 1 || iters < 1 || !sink) return fail(ONEXN_EINVAL, "probe_ffma: blocks, iters >= 1, sink non-NULL");
    onexn::ffma_chain_kernel<<<blocks, 256, 0, static_cast<cudaStream_t>(stream)>>>(iters, 1.0f, sink);
    const cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? ONEXN_OK : fail(ONEXN_ECUDA, "probe_ffma: %s", cudaGetErrorString(e));
}

extern "C" onexn_status onexn_probe_mma_issue(int N, int issuers, int a_tmem, int iters, void *stream)
{
    onexn::clear_error();
    if ((N != 16 && N != 32) || issuers < 1 || issuers > onexn::kProbeWarps || iters < 1)
        return fail(ONEXN_EINVAL, "probe_mma_issue: N in {16, 32}, issuers in 1..8, iters >= 1");
    unsigned int *st = nullptr;
    cudaError_t e = onexn::device_status_ptr(&st);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "probe_mma_issue: %s", cudaGetErrorString(e));
    int sms = 0;
    e = onexn::device_sm_count(&sms);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "probe_mma_issue: %s", cudaGetErrorString(e));
    auto kern = N == 16 ? (a_tmem ? onexn::mma_issue_kernel<16, true> : onexn::mma_issue_kernel<16, false>)
                        : (a_tmem ? onexn::mma_issue_kernel<32, true> : onexn::mma_issue_kernel<32, false>);
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, onexn::kMmaProbeSmem);
    if (e == cudaSuccess) {
        kern<<<sms, onexn::kProbeWarps * 32, onexn::kMmaProbeSmem, static_cast<cudaStream_t>(stream)>>>(
            iters, issuers, st);
        e = cudaGetLastError();
    }
    return e == cudaSuccess ? ONEXN_OK : fail(ONEXN_ECUDA, "probe_mma_issue: %s", cudaGetErrorString(e));
}
