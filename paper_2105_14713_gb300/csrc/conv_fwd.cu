// onexn_conv_fwd: argument checks and kernel selection for the forward
// convolution of a 1xN-pruned layer (Eq. 7).  Launches only; never
// allocates, synchronises or reads device memory from the host.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "onexn_internal.h"

#include <mutex>


using onexn::fail;

// Status word written by kernels that hit a bounded wait (one per device,
// 4 bytes, lives as long as the library is loaded).
__device__ unsigned int g_onexn_status_word;

namespace onexn {

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_dev_mu;
int g_sm_count[kMaxDevices];
unsigned int *g_status_ptr[kMaxDevices];
}  // namespace

cudaError_t device_sm_count(int *sms)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_dev_mu);
    if (g_sm_count[dev] == 0) {
        e = cudaDeviceGetAttribute(&g_sm_count[dev], cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
    }
    *sms = g_sm_count[dev];
    return cudaSuccess;
}

int device_sms_or_default()
{
    int sms = 0;
    return (device_sm_count(&sms) == cudaSuccess && sms > 0) ? sms : 152;
}

cudaError_t device_status_ptr(unsigned int **p)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_dev_mu);
    if (!g_status_ptr[dev]) {
        void *ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_onexn_status_word);
        if (e != cudaSuccess) return e;
        g_status_ptr[dev] = static_cast<unsigned int *>(ptr);
    }
    *p = g_status_ptr[dev];
    return cudaSuccess;
}

}  // namespace onexn

namespace onexn {
namespace detail {

namespace {
bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

// Shape, dtype and flag checks; fills the geometry part of *a.
onexn_status check_shape(const onexn_conv_desc *d, int N, int64_t t, int dtype, unsigned flags,
                         onexn::ConvArgs *a)
{
    if (!d) return fail(ONEXN_EINVAL, "conv: desc is NULL");
    int Ho = 0, Wo = 0;
    onexn_status st = onexn_conv_out_shape(d, &Ho, &Wo);
    if (st != ONEXN_OK) return st;
    if (dtype != ONEXN_F32 && dtype != ONEXN_BF16)
        return fail(ONEXN_EINVAL, "conv: unknown dtype %d", dtype);
    if (N < 1 || d->C_out % N) return fail(ONEXN_EINVAL, "conv: N=%d must divide C_out=%d", N, d->C_out);
    const int64_t K = static_cast<int64_t>(d->KH) * d->KW * d->C_in;
    const int64_t G = d->C_out / N;
    if (K >= (int64_t(1) << 30)) return fail(ONEXN_EINVAL, "conv: index space too large");
    if (t < 0 || t > G * K || t >= (int64_t(1) << 31))
        return fail(ONEXN_EINVAL, "conv: t=%lld outside [0, G*K]", (long long)t);
    const int64_t npix = static_cast<int64_t>(d->B) * Ho * Wo;
    if (npix >= (int64_t(1) << 31) || static_cast<int64_t>(d->B) * d->H * d->W >= (int64_t(1) << 31))
        return fail(ONEXN_EINVAL, "conv: too many pixels for one launch");
    const int cv = dtype == ONEXN_F32 ? 4 : 8;
    if (d->C_in % cv)
        return fail(ONEXN_EINVAL, "conv: C_in=%d must be a multiple of %d for %s", d->C_in, cv,
                    dtype == ONEXN_F32 ? "fp32" : "bf16");
    if (flags & ~(ONEXN_RELU | ONEXN_RELU6 | ONEXN_DECODED | ONEXN_REUSE_DECODE | ONEXN_CHECK_INPUT |
                  ONEXN_ALGO_MASK))
        return fail(ONEXN_EINVAL, "conv: unknown flags");
    a->B = d->B; a->H = d->H; a->W = d->W; a->C = d->C_in;
    a->C_out = d->C_out; a->KH = d->KH; a->KW = d->KW;
    a->sh = d->stride_h; a->sw = d->stride_w; a->ph = d->pad_h; a->pw = d->pad_w;
    a->dh = d->dil_h; a->dw = d->dil_w; a->Ho = Ho; a->Wo = Wo;
    a->N = N; a->t = static_cast<int>(t); a->P_pix = static_cast<int>(npix);
    a->relu = (flags & ONEXN_RELU6) ? 2 : (flags & ONEXN_RELU) ? 1 : 0;
    return ONEXN_OK;
}

// Pointer checks; fills the pointer part of *a.
onexn_status check_pointers(const int32_t *P, const int32_t *I, const void *D, const void *x,
                            void *y, const float *bias, int dtype, onexn::ConvArgs *a)
{
    if (!P) return fail(ONEXN_EINVAL, "conv: P is NULL");
    if (a->t > 0 && (!I || !D)) return fail(ONEXN_EINVAL, "conv: I or D is NULL");
    if (a->P_pix > 0 && (!x || !y)) return fail(ONEXN_EINVAL, "conv: x or y is NULL");
    if (!aligned16(x) || !aligned16(y) || !aligned16(D))
        return fail(ONEXN_EINVAL, "conv: x, y and D must be 16-byte aligned");
    if ((reinterpret_cast<uintptr_t>(bias) & 3u) || (reinterpret_cast<uintptr_t>(P) & 3u) ||
        (reinterpret_cast<uintptr_t>(I) & 3u))
        return fail(ONEXN_EINVAL, "conv: bias, P and I must be 4-byte aligned");
    if (a->P_pix > 0) {
        const size_t es = dtype == ONEXN_F32 ? 4 : 2;
        const uintptr_t x0 = reinterpret_cast<uintptr_t>(x),
                        x1 = x0 + static_cast<size_t>(a->B) * a->H * a->W * a->C * es;
        const uintptr_t y0 = reinterpret_cast<uintptr_t>(y),
                        y1 = y0 + static_cast<size_t>(a->P_pix) * a->C_out * es;
        if (x0 < y1 && y0 < x1) return fail(ONEXN_EINVAL, "conv: x and y overlap");
    }
    a->x = x; a->y = y; a->bias = bias; a->P = P; a->I = I; a->D = D;
    return ONEXN_OK;
}

// Workspace a family needs for these arguments.
size_t workspace_for(unsigned algo, const onexn::ConvArgs &a, int dtype)
{
    if (algo == ONEXN_ALGO_TC) return onexn::tc_workspace_bytes(a, dtype);
    if (algo == ONEXN_ALGO_MMA) return onexn::mma_workspace_bytes(a);
    return 0;
}

size_t workspace_min_for(unsigned algo, const onexn::ConvArgs &a, int dtype)
{
    if (algo == ONEXN_ALGO_TC) return onexn::tc_workspace_min(a, dtype);
    if (algo == ONEXN_ALGO_MMA) return onexn::mma_workspace_bytes(a);
    return 0;
}

// Can the family run this case at all (dtype, shape)?
bool supports(unsigned algo, const onexn::ConvArgs &a, int dtype)
{
    switch (algo) {
    case ONEXN_ALGO_FMA: return true;
    case ONEXN_ALGO_MMA: return dtype == ONEXN_BF16 && onexn::mma_supports(a);
    case ONEXN_ALGO_TC: return onexn::tc_supports(a, dtype);
    default: return false;
    }
}

// Cost model of AUTO.  The machine rates, in ns per multiply-add, are
// fitted to GB300 timings of a 3x3 512->512 layer on 128x14x14 at 50% and
// 90% pruned (fp32 and bf16; the affine fit predicts the 70% point within
// 2%).  The FFMA kernel stages the activations of every 256-pixel x
// 64-column unit whatever is kept (a floor per dense multiply-add, higher
// for small N) and then does only the kept work (t*N weights per pixel),
// faster for wider blocks that share each staged activation.  A unit runs
// on one SM, so a launch with fewer units than SMs (batch-1 layers: a 7x7
// output is one unit of pixels) takes SMs / units times the machine-rate
// time, on pixels and columns padded to whole units (SMs queried from the
// device).  The tensor-core
// family's estimate is tc_cost_ns (conv_tc.cu).  Measured on GB300 at batch
// 1, the FFMA kernel loses to the decoded GEMM on every MobileNet-V2 1x1
// layer from 14x14 down (e.g. 76 vs 17 us on the 7x7 960->160 projection).
namespace {
double fma_floor(int N) { return N >= 4 ? 1.33e-5 : N >= 2 ? 1.66e-5 : 2.67e-5; }
double fma_per_kept(int N) { return N >= 8 ? 3.0e-5 : N >= 4 ? 4.3e-5 : N >= 2 ? 7.2e-5 : 1.44e-4; }
constexpr int kFmaUnitPix = 256, kFmaUnitCols = 64;
constexpr double kFmaFixedNs = 700.0;     // pipeline fill beyond a bare launch

double fma_cost_ns(const onexn::ConvArgs &a)
{
    const int64_t um = (static_cast<int64_t>(a.P_pix) + kFmaUnitPix - 1) / kFmaUnitPix;
    const int64_t un = (a.C_out + kFmaUnitCols - 1) / kFmaUnitCols;
    const int64_t units = um * un;
    const double pix = static_cast<double>(um * kFmaUnitPix);          // padded pixels
    const double col_pad = static_cast<double>(un * kFmaUnitCols) / a.C_out;
    const double K = static_cast<double>(a.KH) * a.KW * a.C;
    const double floor_ns = pix * a.C_out * col_pad * K * fma_floor(a.N);
    const double kept_ns = pix * static_cast<double>(a.t) * a.N * fma_per_kept(a.N);
    const int sms = onexn::device_sms_or_default();
    const double waves = static_cast<double>((units + sms - 1) / sms);
    return (floor_ns + kept_ns) * sms * waves / static_cast<double>(units) + kFmaFixedNs;
}
}  // namespace

// Kernel family for AUTO: the tcgen05 GEMM when its workspace fits and the
// cost model does not expect the FFMA kernel to be faster; otherwise FFMA.
// With ONEXN_DECODED the weights are already decoded: the GEMM.  With
// ONEXN_REUSE_DECODE the caller will keep the decode, so it is left out.
unsigned pick_algo(const onexn::ConvArgs &a, int dtype, unsigned flags, size_t ws_bytes)
{
    const unsigned forced = flags & ONEXN_ALGO_MASK;
    if (forced != ONEXN_ALGO_AUTO) return forced;
    if (flags & ONEXN_DECODED) return ONEXN_ALGO_TC;
    if (!supports(ONEXN_ALGO_TC, a, dtype) || ws_bytes < workspace_min_for(ONEXN_ALGO_TC, a, dtype))
        return ONEXN_ALGO_FMA;
    if (a.t == 0 || a.P_pix == 0) return ONEXN_ALGO_FMA;  // bias only / nothing to do
    const bool amortised = (flags & ONEXN_REUSE_DECODE) != 0;
    return fma_cost_ns(a) < onexn::tc_cost_ns(a, dtype, ws_bytes, amortised) ? ONEXN_ALGO_FMA : ONEXN_ALGO_TC;
}

onexn_status check_algo(unsigned algo, const onexn::ConvArgs &a, int dtype, size_t ws_bytes)
{
    if (algo != ONEXN_ALGO_FMA && algo != ONEXN_ALGO_MMA && algo != ONEXN_ALGO_TC)
        return fail(ONEXN_EINVAL, "conv: unknown algo %u", algo >> ONEXN_ALGO_SHIFT);
    if (!supports(algo, a, dtype))
        return fail(ONEXN_EUNSUPPORTED, "conv: algo %u cannot run this case (dtype/shape)",
                    algo >> ONEXN_ALGO_SHIFT);
    const size_t need = workspace_min_for(algo, a, dtype);
    if (ws_bytes < need)
        return fail(ONEXN_EINVAL, "conv: algo %u needs %zu bytes of workspace, got %zu",
                    algo >> ONEXN_ALGO_SHIFT, need, ws_bytes);
    return ONEXN_OK;
}

cudaError_t launch(unsigned algo, const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes,
                   cudaStream_t st)
{
    if (algo == ONEXN_ALGO_FMA) return launch_fma(a, dtype, st);
    if (algo == ONEXN_ALGO_MMA) return launch_mma(a, workspace, ws_bytes, st);
    return launch_tc(a, dtype, workspace, ws_bytes, st);
}

}  // namespace detail
}  // namespace onexn

namespace onexn {

// Checked mode: the BSR lists of Sec. 3.4 as the kernels assume them --
// P[0] = 0, P[G] = t, P non-decreasing; within every group I strictly
// increasing and inside [0, K).  One thread per group; every read is
// clamped to P[0..G] and I[0..t), so a malformed list is reported through
// the status word instead of being read out of bounds.
__global__ void validate_bsr_kernel(const int32_t *__restrict__ P, const int32_t *__restrict__ I, int G, int t,
                                    int K, unsigned int *status)
{
    const int g = blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= G) return;
    const int p0 = __ldg(P + g), p1 = __ldg(P + g + 1);
    bool ok = p0 >= 0 && p1 <= t && p0 <= p1;
    if (g == 0 && p0 != 0) ok = false;
    if (g == G - 1 && p1 != t) ok = false;
    const int z0 = clampi(p0, 0, t), z1 = clampi(p1, z0, t);
    int prev = -1;
    for (int z = z0; z < z1 && ok; ++z) {
        const int k = __ldg(I + z);
        if (k <= prev || k >= K) ok = false;
        prev = k;
    }
    if (!ok) atomicOr(status, kStatusBadInput);
}

namespace detail {
cudaError_t launch_validate(const ConvArgs &a, cudaStream_t st)
{
    const int G = a.C_out / a.N;
    if (G == 0) return cudaSuccess;
    validate_bsr_kernel<<<(G + 127) / 128, 128, 0, st>>>(a.P, a.I, G, a.t, a.KH * a.KW * a.C, a.status);
    return cudaGetLastError();
}
}  // namespace detail
}  // namespace onexn

using namespace onexn::detail;

extern "C" onexn_status onexn_conv_algo(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                                        unsigned flags, size_t workspace_bytes, unsigned *algo)
{
    onexn::clear_error();
    if (!algo) return fail(ONEXN_EINVAL, "conv_algo: algo is NULL");
    onexn::ConvArgs a{};
    onexn_status st = check_shape(desc, N, t, dtype, flags, &a);
    if (st != ONEXN_OK) return st;
    const unsigned al = pick_algo(a, dtype, flags, workspace_bytes);
    st = check_algo(al, a, dtype, workspace_bytes);
    if (st != ONEXN_OK) return st;
    if ((flags & ONEXN_DECODED) && al != ONEXN_ALGO_TC)
        return fail(ONEXN_EINVAL, "conv: ONEXN_DECODED needs the tc family");
    *algo = al;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_tc_form(const onexn_conv_desc *desc, int N, int64_t t, int dtype, int *form)
{
    onexn::clear_error();
    if (!form) return fail(ONEXN_EINVAL, "conv_tc_form: form is NULL");
    onexn::ConvArgs a{};
    onexn_status st = check_shape(desc, N, t, dtype, 0, &a);
    if (st != ONEXN_OK) return st;
    *form = onexn::tc_gemm_form(a, dtype);
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_halo_geometry(const onexn_conv_desc *desc, int N, int64_t t, int *geom,
                                                 uint32_t *taps, uint32_t *phases)
{
    onexn::clear_error();
    if (!geom || !taps || !phases) return fail(ONEXN_EINVAL, "conv_halo_geometry: NULL output");
    onexn::ConvArgs a{};
    onexn_status st = check_shape(desc, N, t, ONEXN_BF16, 0, &a);
    if (st != ONEXN_OK) return st;
    if (!onexn::halo_streamed_geometry(a, geom, taps, phases))
        return fail(ONEXN_EUNSUPPORTED, "conv_halo_geometry: no streamed halo plan for this layer");
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_workspace_size(const onexn_conv_desc *desc, int N, int64_t t,
                                                  int dtype, unsigned flags, size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "conv_workspace_size: bytes is NULL");
    onexn::ConvArgs a{};
    onexn_status st = check_shape(desc, N, t, dtype, flags, &a);
    if (st != ONEXN_OK) return st;
    const unsigned forced = flags & ONEXN_ALGO_MASK;
    size_t need = 0;
    if (forced == ONEXN_ALGO_AUTO) {
        for (unsigned al : {ONEXN_ALGO_FMA, ONEXN_ALGO_MMA, ONEXN_ALGO_TC})
            if (supports(al, a, dtype) && workspace_for(al, a, dtype) > need) need = workspace_for(al, a, dtype);
    } else {
        if (!supports(forced, a, dtype))
            return fail(ONEXN_EUNSUPPORTED, "conv: algo %u cannot run this case", forced >> ONEXN_ALGO_SHIFT);
        need = workspace_for(forced, a, dtype);
    }
    *bytes = need;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_fwd_ex(const onexn_conv_desc *desc, const int32_t *P,
                                          const int32_t *I, const void *D, int N, int64_t t,
                                          const void *x, void *y, const float *bias, const void *residual,
                                          int dtype, unsigned flags, void *workspace, size_t workspace_bytes,
                                          void *stream)
{
    onexn::clear_error();
    onexn::ConvArgs a{};
    onexn_status st = check_shape(desc, N, t, dtype, flags, &a);
    if (st != ONEXN_OK) return st;
    st = check_pointers(P, I, D, x, y, bias, dtype, &a);
    if (st != ONEXN_OK) return st;
    if (residual) {
        if (reinterpret_cast<uintptr_t>(residual) & 15u)
            return fail(ONEXN_EINVAL, "conv: residual must be 16-byte aligned");
        const size_t yb = static_cast<size_t>(a.P_pix) * a.C_out * (dtype == ONEXN_F32 ? 4 : 2);
        const uintptr_t r0 = reinterpret_cast<uintptr_t>(residual), y0 = reinterpret_cast<uintptr_t>(y);
        if (r0 != y0 && r0 < y0 + yb && y0 < r0 + yb)
            return fail(ONEXN_EINVAL, "conv: residual overlaps y without being y");
        a.residual = residual;
    }
    if (!workspace) workspace_bytes = 0;
    if (reinterpret_cast<uintptr_t>(workspace) & 255u)
        return fail(ONEXN_EINVAL, "conv: workspace must be 256-byte aligned");
    const unsigned algo = pick_algo(a, dtype, flags, workspace_bytes);
    st = check_algo(algo, a, dtype, workspace_bytes);
    if (st != ONEXN_OK) return st;
    const bool decoded = (flags & ONEXN_DECODED) != 0;
    if (decoded && algo != ONEXN_ALGO_TC) return fail(ONEXN_EINVAL, "conv: ONEXN_DECODED needs the tc family");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = onexn::device_status_ptr(&a.status);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv: status word: %s", cudaGetErrorString(e));
    if ((flags & ONEXN_CHECK_INPUT) && (e = launch_validate(a, s)) != cudaSuccess)
        return fail(ONEXN_ECUDA, "conv: validation launch failed: %s", cudaGetErrorString(e));
    e = decoded ? tc_gemm(a, dtype, workspace, workspace_bytes, s) : launch(algo, a, dtype, workspace, workspace_bytes, s);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}

extern "C" onexn_status onexn_dwproj_fwd(const onexn_conv_desc *dw_desc, const float *W_dw, const float *b_dw,
                                         const int32_t *P, const int32_t *I, const void *D, int N, int64_t t,
                                         int C_out, const void *h, void *y, const float *bias, const void *residual,
                                         int dtype, unsigned flags, void *workspace, size_t workspace_bytes,
                                         void *stream)
{
    onexn::clear_error();
    if (!dw_desc) return fail(ONEXN_EINVAL, "dwproj: dw_desc is NULL");
    const onexn_conv_desc &d = *dw_desc;
    if (d.C_in != d.C_out || d.KH != 3 || d.KW != 3 || d.pad_h != 1 || d.pad_w != 1 || d.dil_h != 1 ||
        d.dil_w != 1 || d.stride_h != d.stride_w || (d.stride_h != 1 && d.stride_h != 2))
        return fail(ONEXN_EINVAL, "dwproj: the depthwise must be 3x3, pad 1, stride 1 or 2, C_in == C_out");
    if (dtype != ONEXN_F32) return fail(ONEXN_EUNSUPPORTED, "dwproj: the fused form runs fp32 only");
    int Ho = 0, Wo = 0;
    onexn_status st = onexn_conv_out_shape(dw_desc, &Ho, &Wo);
    if (st != ONEXN_OK) return st;
    const unsigned forced = flags & ONEXN_ALGO_MASK;
    if (forced != ONEXN_ALGO_AUTO && forced != ONEXN_ALGO_TC)
        return fail(ONEXN_EINVAL, "dwproj: only the tensor-core family runs the fused form");
    // the projection: a 1x1 layer on the depthwise's output grid
    onexn_conv_desc pd{};
    pd.B = d.B; pd.H = Ho; pd.W = Wo; pd.C_in = d.C_in; pd.C_out = C_out;
    pd.KH = 1; pd.KW = 1; pd.stride_h = 1; pd.stride_w = 1; pd.pad_h = 0; pd.pad_w = 0; pd.dil_h = 1; pd.dil_w = 1;
    onexn::ConvArgs a{};
    st = check_shape(&pd, N, t, dtype, (flags & ~ONEXN_ALGO_MASK) | ONEXN_ALGO_TC, &a);
    if (st != ONEXN_OK) return st;
    st = check_pointers(P, I, D, h, y, bias, dtype, &a);
    if (st != ONEXN_OK) return st;
    if (a.P_pix > 0 && !W_dw) return fail(ONEXN_EINVAL, "dwproj: W_dw is NULL");
    if ((reinterpret_cast<uintptr_t>(W_dw) & 15u) || (reinterpret_cast<uintptr_t>(b_dw) & 3u))
        return fail(ONEXN_EINVAL, "dwproj: W_dw must be 16-byte and b_dw 4-byte aligned");
    if (!supports(ONEXN_ALGO_TC, a, dtype))
        return fail(ONEXN_EUNSUPPORTED, "dwproj: the tensor-core family cannot run this projection");
    {
        const uintptr_t h0 = reinterpret_cast<uintptr_t>(h), y0 = reinterpret_cast<uintptr_t>(y);
        const size_t hb = static_cast<size_t>(d.B) * d.H * d.W * d.C_in * 4, yb = static_cast<size_t>(a.P_pix) * C_out * 4;
        if (a.P_pix > 0 && h0 < y0 + yb && y0 < h0 + hb) return fail(ONEXN_EINVAL, "dwproj: h and y overlap");
    }
    if (residual) {
        if (reinterpret_cast<uintptr_t>(residual) & 15u)
            return fail(ONEXN_EINVAL, "dwproj: residual must be 16-byte aligned");
        const size_t yb = static_cast<size_t>(a.P_pix) * a.C_out * 4;
        const uintptr_t r0 = reinterpret_cast<uintptr_t>(residual), y0 = reinterpret_cast<uintptr_t>(y);
        if (r0 != y0 && r0 < y0 + yb && y0 < r0 + yb)
            return fail(ONEXN_EINVAL, "dwproj: residual overlaps y without being y");
        a.residual = residual;
    }
    if (!workspace) workspace_bytes = 0;
    if (reinterpret_cast<uintptr_t>(workspace) & 255u)
        return fail(ONEXN_EINVAL, "dwproj: workspace must be 256-byte aligned");
    st = check_algo(ONEXN_ALGO_TC, a, dtype, workspace_bytes);
    if (st != ONEXN_OK) return st;
    if (a.P_pix == 0) return ONEXN_OK;
    a.dw_x = static_cast<const float *>(h);
    a.dw_w = W_dw;
    a.dw_b = b_dw;
    a.dw_H = d.H; a.dw_W = d.W; a.dw_s = d.stride_h;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = onexn::device_status_ptr(&a.status);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "dwproj: status word: %s", cudaGetErrorString(e));
    e = (flags & ONEXN_DECODED) ? onexn::tc_gemm(a, dtype, workspace, workspace_bytes, s)
                                : onexn::launch_tc(a, dtype, workspace, workspace_bytes, s);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "dwproj: launch failed: %s", cudaGetErrorString(e));
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_fwd(const onexn_conv_desc *desc, const int32_t *P,
                                       const int32_t *I, const void *D, int N, int64_t t,
                                       const void *x, void *y, const float *bias, int dtype,
                                       unsigned flags, void *workspace, size_t workspace_bytes,
                                       void *stream)
{
    return onexn_conv_fwd_ex(desc, P, I, D, N, t, x, y, bias, nullptr, dtype, flags, workspace, workspace_bytes,
                             stream);
}

namespace onexn {

// Waits on a fresh mbarrier that nothing signals: the bounded wait every
// library kernel uses runs out (about 2^31 SM cycles) and the kernel reports
// it in the status word, as a kernel whose pipeline stalled would.
__global__ void selftest_wait_kernel(unsigned int *status)
{
    __shared__ __align__(8) unsigned long long bar;
    const uint32_t b = static_cast<uint32_t>(__cvta_generic_to_shared(&bar));
    mbar_init(b, 1);
    fence_mbar_init();
    if (!mbar_wait(b, 0)) atomicOr(status, kStatusTimeout);
    asm volatile("mbarrier.inval.shared::cta.b64 [%0];\n" ::"r"(b) : "memory");
}

}  // namespace onexn

extern "C" onexn_status onexn_selftest_timeout(void *stream)
{
    onexn::clear_error();
    unsigned int *p = nullptr;
    cudaError_t e = onexn::device_status_ptr(&p);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "selftest_timeout: status word: %s", cudaGetErrorString(e));
    onexn::selftest_wait_kernel<<<1, 1, 0, static_cast<cudaStream_t>(stream)>>>(p);
    e = cudaGetLastError();
    return e == cudaSuccess ? ONEXN_OK : fail(ONEXN_ECUDA, "selftest_timeout: %s", cudaGetErrorString(e));
}

extern "C" onexn_status onexn_device_status(int clear, int *status)
{
    onexn::clear_error();
    if (!status) return fail(ONEXN_EINVAL, "device_status: status is NULL");
    unsigned int *p = nullptr;
    cudaError_t e = onexn::device_status_ptr(&p);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    unsigned int w = 0;
    if (e == cudaSuccess) e = cudaMemcpy(&w, p, sizeof(w), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && clear) e = cudaMemset(p, 0, sizeof(w));
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "device_status: %s", cudaGetErrorString(e));
    *status = (w & onexn::kStatusBadInput) ? ONEXN_EDEVICE : (w & onexn::kStatusTimeout) ? ONEXN_ETIMEOUT : ONEXN_OK;
    return ONEXN_OK;
}
