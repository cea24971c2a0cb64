// onexn_conv_fwd_host: the forward convolution of a 1xN-pruned layer (Eq. 7)
// on activations that live in host memory.
//
// The batch is cut into chunks of whole images.  Each chunk's input is copied
// to a device slot, convolved into an output slot and copied back, on three
// kinds of streams so that the copy engines and the SMs work at the same time:
//   in-stream:       H2D of chunk i into x slot i % S   (after the GEMM of
//                    chunk i - S has read that slot)
//   compute streams: the GEMM of chunk i on stream i % 2 (after its H2D and
//                    after the D2H of chunk i - S has read its y slot); two
//                    streams let the next chunk's persistent kernel take SMs
//                    as the previous one's tail retires
//   out-stream:      D2H of chunk i (after its GEMM)
// (More streams per copy direction, and chunks of 2 to 16 MiB, measured no
// faster on GB300: host-link copies in both directions were the bound.)
// The tensor-core family decodes the weights once per call, before the first
// GEMM.  Work on the caller's stream before the call happens before the
// first copy; the caller's stream waits for the last copy, so synchronising
// it makes y_host valid.  Successive calls on different caller streams (and
// with different workspaces) overlap: the next layer's input copies run
// while this one computes and copies out.  Streams and events are created
// once per device and reused; a per-device mutex serialises the enqueueing.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "onexn_internal.h"

#include <mutex>

using onexn::fail;

namespace {

constexpr int kSlots = 3;                       // x / y device slots per call
constexpr int kCopyStreams = 1;                 // streams per copy direction
constexpr size_t kChunkTarget = size_t(8) << 20;  // aim for ~8 MiB of input per chunk
constexpr int kMaxChunks = 8;
constexpr int kMaxDev = 64;

size_t round256(size_t v) { return (v + 255) & ~size_t(255); }

struct HostPipe {
    cudaStream_t in[kCopyStreams] = {}, out[kCopyStreams] = {}, cmp[2] = {nullptr, nullptr};
    cudaEvent_t start = nullptr, dec = nullptr, end[kCopyStreams] = {};
    cudaEvent_t ev_in[kSlots] = {}, ev_cmp[kSlots] = {}, ev_out[kSlots] = {};
    std::mutex mu;
    bool ready = false;
};
HostPipe g_pipe[kMaxDev];
std::mutex g_pipe_mu;

cudaError_t pipe_for_current_device(HostPipe **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDev) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_pipe_mu);
    HostPipe &p = g_pipe[dev];
    if (!p.ready) {
        const unsigned sf = cudaStreamNonBlocking;
        const unsigned ef = cudaEventDisableTiming;
        for (cudaStream_t *s : {&p.cmp[0], &p.cmp[1]})
            if (!*s && (e = cudaStreamCreateWithFlags(s, sf)) != cudaSuccess) return e;
        for (int i = 0; i < kCopyStreams; ++i)
            for (cudaStream_t *s : {&p.in[i], &p.out[i]})
                if (!*s && (e = cudaStreamCreateWithFlags(s, sf)) != cudaSuccess) return e;
        for (cudaEvent_t *v : {&p.start, &p.dec})
            if (!*v && (e = cudaEventCreateWithFlags(v, ef)) != cudaSuccess) return e;
        for (int i = 0; i < kCopyStreams; ++i)
            if (!p.end[i] && (e = cudaEventCreateWithFlags(&p.end[i], ef)) != cudaSuccess) return e;
        for (int i = 0; i < kSlots; ++i) {
            cudaEvent_t *vs[3] = {&p.ev_in[i], &p.ev_cmp[i], &p.ev_out[i]};
            for (cudaEvent_t *v : vs)
                if (!*v && (e = cudaEventCreateWithFlags(v, ef)) != cudaSuccess) return e;
        }
        p.ready = true;
    }
    *out = &p;
    return cudaSuccess;
}

// Chunking of a batch of B images of x_image bytes each.
int chunk_images(int B, size_t x_image)
{
    if (B <= 0) return 1;
    size_t n = (static_cast<size_t>(B) * x_image + kChunkTarget / 2) / kChunkTarget;
    if (n < 1) n = 1;
    if (n > static_cast<size_t>(kMaxChunks)) n = kMaxChunks;
    if (n > static_cast<size_t>(B)) n = B;
    return static_cast<int>((B + n - 1) / n);
}

struct HostPlan {
    onexn::ConvArgs a{};       // whole-batch arguments (geometry only)
    unsigned algo = 0;
    int chunk = 1;             // images per chunk
    size_t es = 4;             // element size
    size_t x_image = 0, y_image = 0;   // bytes per image
    size_t kernel_ws = 0, x_slot = 0, y_slot = 0;
    size_t total() const { return round256(kernel_ws) + kSlots * (x_slot + y_slot); }
};

onexn_status plan(const onexn_conv_desc *desc, int N, int64_t t, int dtype, unsigned flags, HostPlan *hp)
{
    if (flags & (ONEXN_DECODED | ONEXN_REUSE_DECODE))      // every call decodes into its own workspace
        return onexn::fail(ONEXN_EINVAL, "conv_host: ONEXN_DECODED / ONEXN_REUSE_DECODE are not accepted here");
    onexn_status st = onexn::detail::check_shape(desc, N, t, dtype, flags, &hp->a);
    if (st != ONEXN_OK) return st;
    const onexn::ConvArgs &a = hp->a;
    hp->es = dtype == ONEXN_F32 ? 4 : 2;
    hp->x_image = static_cast<size_t>(a.H) * a.W * a.C * hp->es;
    hp->y_image = static_cast<size_t>(a.Ho) * a.Wo * a.C_out * hp->es;
    hp->chunk = chunk_images(a.B, hp->x_image);
    hp->x_slot = round256(hp->chunk * hp->x_image);
    hp->y_slot = round256(hp->chunk * hp->y_image);
    // The family: as onexn_conv_fwd would choose for the whole batch when
    // given the workspace the family needs.
    const unsigned forced = flags & ONEXN_ALGO_MASK;
    size_t ws = 0;
    for (unsigned al : {ONEXN_ALGO_FMA, ONEXN_ALGO_MMA, ONEXN_ALGO_TC})
        if ((forced == ONEXN_ALGO_AUTO || forced == al) && onexn::detail::supports(al, a, dtype) &&
            onexn::detail::workspace_min_for(al, a, dtype) > ws)
            ws = onexn::detail::workspace_min_for(al, a, dtype);
    hp->algo = onexn::detail::pick_algo(a, dtype, flags, ws);
    st = onexn::detail::check_algo(hp->algo, a, dtype, ws);
    if (st != ONEXN_OK) return st;
    // chunk GEMMs may run concurrently on the two compute streams, so they
    // get no shared stream-K space: the decoded weights only
    hp->kernel_ws = onexn::detail::workspace_min_for(hp->algo, a, dtype);
    return ONEXN_OK;
}

}  // namespace

extern "C" onexn_status onexn_conv_host_workspace_size(const onexn_conv_desc *desc, int N, int64_t t,
                                                       int dtype, unsigned flags, size_t *bytes)
{
    onexn::clear_error();
    if (!bytes) return fail(ONEXN_EINVAL, "conv_host_workspace_size: bytes is NULL");
    HostPlan hp;
    const onexn_status st = plan(desc, N, t, dtype, flags, &hp);
    if (st != ONEXN_OK) return st;
    *bytes = hp.total();
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_fwd_host(const onexn_conv_desc *desc, const int32_t *P,
                                            const int32_t *I, const void *D, int N, int64_t t,
                                            const void *x_host, void *y_host, const float *bias,
                                            int dtype, unsigned flags, void *workspace,
                                            size_t workspace_bytes, void *stream)
{
    onexn::clear_error();
    HostPlan hp;
    onexn_status st = plan(desc, N, t, dtype, flags, &hp);
    if (st != ONEXN_OK) return st;
    onexn::ConvArgs a = hp.a;
    if (a.B > 0 && (!x_host || !y_host)) return fail(ONEXN_EINVAL, "conv_host: x_host or y_host is NULL");
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u))
        return fail(ONEXN_EINVAL, "conv_host: workspace must be non-NULL and 256-byte aligned");
    if (workspace_bytes < hp.total())
        return fail(ONEXN_EINVAL, "conv_host: needs %zu bytes of workspace, got %zu", hp.total(),
                    workspace_bytes);
    // device-pointer checks on one chunk in the first slots (they stand for
    // every chunk)
    unsigned char *ws = static_cast<unsigned char *>(workspace);
    unsigned char *xs = ws + round256(hp.kernel_ws);
    unsigned char *ys = xs + kSlots * hp.x_slot;
    onexn::ConvArgs c0 = a;
    c0.B = a.B < hp.chunk ? a.B : hp.chunk;
    c0.P_pix = c0.B * a.Ho * a.Wo;
    st = onexn::detail::check_pointers(P, I, D, xs, ys, bias, dtype, &c0);
    if (st != ONEXN_OK) return st;
    a.P = c0.P;
    a.I = c0.I;
    a.D = c0.D;
    a.bias = c0.bias;
    if (a.B == 0) return ONEXN_OK;
    cudaError_t e = onexn::device_status_ptr(&a.status);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_host: status word: %s", cudaGetErrorString(e));
    HostPipe *pp = nullptr;
    e = pipe_for_current_device(&pp);
    if (e != cudaSuccess) return fail(ONEXN_ECUDA, "conv_host: streams: %s", cudaGetErrorString(e));
    HostPipe &p = *pp;
    cudaStream_t caller = static_cast<cudaStream_t>(stream);

    std::lock_guard<std::mutex> lk(p.mu);
#define ONEXN_TRY(call)                                                                        \
    do {                                                                                       \
        const cudaError_t e_ = (call);                                                         \
        if (e_ != cudaSuccess)                                                                 \
            return fail(ONEXN_ECUDA, "conv_host: %s: %s", #call, cudaGetErrorString(e_));      \
    } while (0)
    ONEXN_TRY(cudaEventRecord(p.start, caller));
    for (cudaStream_t s : {p.cmp[0], p.cmp[1]}) ONEXN_TRY(cudaStreamWaitEvent(s, p.start, 0));
    for (int k = 0; k < kCopyStreams; ++k) {
        ONEXN_TRY(cudaStreamWaitEvent(p.in[k], p.start, 0));
        ONEXN_TRY(cudaStreamWaitEvent(p.out[k], p.start, 0));
    }
    if (hp.algo == ONEXN_ALGO_TC) {
        ONEXN_TRY(onexn::tc_decode(a, dtype, ws, hp.kernel_ws, p.cmp[0]));
        ONEXN_TRY(cudaEventRecord(p.dec, p.cmp[0]));
        ONEXN_TRY(cudaStreamWaitEvent(p.cmp[1], p.dec, 0));
    }
    const unsigned char *xh = static_cast<const unsigned char *>(x_host);
    unsigned char *yh = static_cast<unsigned char *>(y_host);
    const int n_chunks = (a.B + hp.chunk - 1) / hp.chunk;
    for (int i = 0; i < n_chunks; ++i) {
        const int slot = i % kSlots;
        const int b0 = i * hp.chunk;
        const int nb = a.B - b0 < hp.chunk ? a.B - b0 : hp.chunk;
        unsigned char *xd = xs + slot * hp.x_slot;
        unsigned char *yd = ys + slot * hp.y_slot;
        cudaStream_t cs = p.cmp[i & 1];
        cudaStream_t in = p.in[i % kCopyStreams], out = p.out[i % kCopyStreams];
        // in: the slot is free once the GEMM of chunk i - kSlots has run
        if (i >= kSlots) ONEXN_TRY(cudaStreamWaitEvent(in, p.ev_cmp[slot], 0));
        ONEXN_TRY(cudaMemcpyAsync(xd, xh + b0 * hp.x_image, nb * hp.x_image, cudaMemcpyHostToDevice, in));
        ONEXN_TRY(cudaEventRecord(p.ev_in[slot], in));
        // compute
        ONEXN_TRY(cudaStreamWaitEvent(cs, p.ev_in[slot], 0));
        if (i >= kSlots) ONEXN_TRY(cudaStreamWaitEvent(cs, p.ev_out[slot], 0));
        onexn::ConvArgs c = a;
        c.B = nb;
        c.P_pix = nb * a.Ho * a.Wo;
        c.x = xd;
        c.y = yd;
        if (hp.algo == ONEXN_ALGO_TC)
            ONEXN_TRY(onexn::tc_gemm(c, dtype, ws, hp.kernel_ws, cs));
        else
            ONEXN_TRY(onexn::detail::launch(hp.algo, c, dtype, ws, hp.kernel_ws, cs));
        ONEXN_TRY(cudaEventRecord(p.ev_cmp[slot], cs));
        // out
        ONEXN_TRY(cudaStreamWaitEvent(out, p.ev_cmp[slot], 0));
        ONEXN_TRY(cudaMemcpyAsync(yh + b0 * hp.y_image, yd, nb * hp.y_image, cudaMemcpyDeviceToHost, out));
        ONEXN_TRY(cudaEventRecord(p.ev_out[slot], out));
    }
    // every D2H follows its GEMM, and each GEMM its H2D: the ends of the
    // out-streams cover the whole call
    for (int k = 0; k < kCopyStreams; ++k) {
        ONEXN_TRY(cudaEventRecord(p.end[k], p.out[k]));
        ONEXN_TRY(cudaStreamWaitEvent(caller, p.end[k], 0));
    }
#undef ONEXN_TRY
    return ONEXN_OK;
}
