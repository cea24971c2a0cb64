// onexn_conv_fwd_noalloc: the tensor-core convolution for callers that
// cannot allocate device memory.
//
// The tensor-core family needs scratch space for the decoded weight matrix
// (C_out x KH*KW*C_in bf16 values, or twice that many fp32 values for fp32
// layers).  onexn_conv_fwd expects the caller to
// provide it.  Some callers cannot: code that runs while a CUDA stream is
// being captured into a graph (a cudaMalloc there breaks the capture), hosts
// that forbid allocation after start-up so that latency stays predictable,
// and plug-ins that only see raw pointers handed to them by a framework that
// owns all device memory.  This entry point serves them: its scratch is one
// fixed array that lives in the library's own device image, so a call never
// allocates or frees anything.
//
// Costs and limits:
//  * Every GPU that loads the library holds kNoAllocScratchBytes (8 MiB) of
//    device memory for this array until the process exits.
//  * Layers whose decoded weights exceed that size are rejected with
//    ONEXN_EINVAL; use onexn_conv_fwd with a workspace for them.
//  * All calls share the one array.  Calls that overlap on the GPU (on
//    different streams, or from different host threads) race on it and may
//    produce wrong results; serialise them.
//  * Nothing in the array has to start at zero: the decode step of each
//    call writes every element of the weight region the call uses (a kept
//    weight or zero) and lowers the stream-K flags before the GEMM reads
//    them; the GEMM reads a stream-K partial slot only after its writer
//    raised that slot's flag in the same call.  Contents left by the
//    previous call are never read.
//  * The device address of the array is looked up once per device, on the
//    first call made with that device current (cudaGetSymbolAddress).  Make
//    that first call before any stream capture begins.
#include "conv_dispatch.h"
#include "onexn_internal.h"

#include <cuda_runtime.h>

#include <mutex>

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;   // 8 MiB
constexpr int kMaxDev = 64;

// Host code must not use this name as a device address: on the host it is
// only a stand-in for the symbol.  The device address comes from
// cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
void *g_scratch_ptr[kMaxDev];

// Device address of the scratch array on the current device (set up once).
onexn_status scratch_ptr(void **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return onexn::fail(ONEXN_ECUDA, "conv_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDev) return onexn::fail(ONEXN_EUNSUPPORTED, "conv_noalloc: device %d", dev);
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return onexn::fail(ONEXN_ECUDA, "conv_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return ONEXN_OK;
}

}  // namespace

extern "C" onexn_status onexn_conv_fwd_noalloc(const onexn_conv_desc *desc, const int32_t *P,
                                               const int32_t *I, const void *D, int N, int64_t t,
                                               const void *x, void *y, const float *bias, int dtype,
                                               unsigned flags, void *stream)
{
    onexn::clear_error();
    if ((flags & ONEXN_ALGO_MASK) != ONEXN_ALGO_AUTO && (flags & ONEXN_ALGO_MASK) != ONEXN_ALGO_TC)
        return onexn::fail(ONEXN_EINVAL, "conv_noalloc: only the tensor-core family runs here");
    if (flags & (ONEXN_DECODED | ONEXN_REUSE_DECODE))      // the scratch is shared by every layer
        return onexn::fail(ONEXN_EINVAL, "conv_noalloc: ONEXN_DECODED / ONEXN_REUSE_DECODE are not accepted here");
    const unsigned f = (flags & ~ONEXN_ALGO_MASK) | ONEXN_ALGO_TC;
    onexn::ConvArgs a{};
    onexn_status st = onexn::detail::check_shape(desc, N, t, dtype, f, &a);
    if (st != ONEXN_OK) return st;
    if (!onexn::detail::supports(ONEXN_ALGO_TC, a, dtype))
        return onexn::fail(ONEXN_EUNSUPPORTED, "conv_noalloc: the tensor-core family cannot run this case");
    // the decoded weights must fit.  The whole scratch is passed on as the
    // workspace: when the decoded weights plus the stream-K partial slots
    // and flags also fit in it, the GEMM balances its last round of tiles
    // there too (each call's decode lowers the flags before the GEMM reads
    // them, so nothing a previous call left behind is trusted)
    const size_t need = onexn::detail::workspace_min_for(ONEXN_ALGO_TC, a, dtype);
    if (need > kNoAllocScratchBytes)
        return onexn::fail(ONEXN_EINVAL,
                           "conv_noalloc: decoded weights need %zu bytes, more than the fixed %zu-byte "
                           "scratch; call onexn_conv_fwd with a workspace instead",
                           need, kNoAllocScratchBytes);
    void *scratch = nullptr;
    st = scratch_ptr(&scratch);
    if (st != ONEXN_OK) return st;
    return onexn_conv_fwd(desc, P, I, D, N, t, x, y, bias, dtype, f, scratch, kNoAllocScratchBytes, stream);
}
