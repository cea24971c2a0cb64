/*
 * onexn.h -- C ABI of the GB300 (sm_103a) 1xN-pruned convolution library.
 *
 * 1xN pruning (Lin et al., "1xN Pattern for Pruning Convolutional Neural
 * Networks") groups the weights of a layer W in R^{n x m x h x w}
 * (n = C_out, m = C_in, h x w = KH x KW, Sec. 3.1) into blocks of N
 * consecutive output channels that share one input index, keeps the blocks
 * with the largest l1 norms (Sec. 3.2, Eq. 4-5), optionally re-orders the
 * filters by l1 norm first (Sec. 3.3), stores the kept blocks in a BSR
 * layout (D, I, P) (Sec. 3.4) and computes the layer output block by block
 * (Eq. 7).  This header is the whole public surface: plain C types, host or
 * device pointers, and sizes.
 *
 * Conventions used by every call
 * ------------------------------
 *  - Weights W are host fp32 in OIHW order: W[o][c][kh][kw].
 *  - Index space.  A block is one (col-group g, input index k), where
 *    g in [0, G), G = C_out / N, and k = (kh*KW + kw)*C_in + c in [0, K),
 *    K = KH*KW*C_in ("tap-major": it matches the NHWC activation layout).
 *    This is the per-(c, kh, kw) block granularity (ONEXN_GRAN_TAP).
 *    ONEXN_GRAN_KERNEL is the paper's own block of Sec. 3.2, one block per
 *    (g, c) holding N whole KH x KW kernels; a kept (g, c) keeps all KH*KW
 *    indices k of channel c.  The two coincide for 1x1 layers.
 *  - mask is uint8 [G][K] (1 = kept), the transpose of the paper's
 *    T in {0,1}^{m x n/N} expanded to the index space.
 *  - BSR (Sec. 3.4), 0-based: P int32 [G+1] with P[0] = 0 and P[G] = t,
 *    I int32 [t] (strictly increasing inside each col-group), D [t][N]
 *    (the N weights of a kept block stored contiguously), fp32 or bf16.
 *  - Activations are NHWC: x[b][h][w][c]; outputs y[b][ho][wo][o].
 *  - Every call returns an onexn_status; nothing else crosses the ABI.
 *    On failure onexn_last_error() returns a message (thread-local, valid
 *    until the next call on the same thread).  Calls allocate nothing that
 *    outlives them and take no ownership of caller buffers.
 */
#ifndef ONEXN_H
#define ONEXN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    ONEXN_OK = 0,
    ONEXN_EINVAL = 1,        /* bad argument: shape, null pointer, range, alignment */
    ONEXN_EUNSUPPORTED = 2,  /* valid request that no kernel here implements */
    ONEXN_ENOMEM = 3,        /* a host allocation failed */
    ONEXN_ECUDA = 4,         /* a CUDA runtime call or kernel launch failed */
    ONEXN_EDEVICE = 5,       /* a kernel reported a bad input through its status word */
    ONEXN_ETIMEOUT = 6       /* a bounded device-side wait ran out */
} onexn_status;

typedef enum { ONEXN_F32 = 0, ONEXN_BF16 = 1 } onexn_dtype;

typedef enum { ONEXN_GRAN_TAP = 0, ONEXN_GRAN_KERNEL = 1 } onexn_granularity;

/* onexn_conv_fwd flags */
#define ONEXN_RELU 0x1u               /* y = max(y, 0) after the bias (and residual) */
#define ONEXN_RELU6 0x2u              /* y = min(max(y, 0), 6) (MobileNet-V2); wins over RELU */
/* ONEXN_DECODED (onexn_conv_fwd / _ex only): the workspace already holds this
 * layer's decoded weights, written by an earlier ONEXN_ALGO_TC call with the
 * same P, I, D, N, t, dtype and geometry on the same workspace, which the
 * caller has ordered before this one (same stream, or an event); the call
 * skips the decode and runs the GEMM alone.  It implies the tc family (AUTO
 * resolves to it; another forced ALGO is EINVAL).  Weights that changed since,
 * a workspace another layer used in between, or a previous call on it that
 * reported ONEXN_ETIMEOUT through onexn_device_status: run once without the
 * flag first. */
#define ONEXN_DECODED 0x10u
/* ONEXN_REUSE_DECODE (onexn_conv_fwd / _ex / _algo / _workspace_size): a hint
 * for AUTO that the caller keeps the workspace's decoded weights and passes
 * ONEXN_DECODED on later calls, so the one-time decode is left out of the
 * comparison of the families.  It changes nothing else. */
#define ONEXN_REUSE_DECODE 0x20u
/* ONEXN_ACCUMULATE (onexn_conv_bwd_data only): dx += the gradient instead of
 * dx = the gradient (a layer whose input also feeds another branch). */
#define ONEXN_ACCUMULATE 0x40u
/* ONEXN_CHECK_INPUT (onexn_conv_fwd / _ex): checked mode.  Before the
 * convolution a validation kernel checks the device BSR lists as Sec. 3.4
 * defines them (P[0] = 0, P[G] = t, P non-decreasing, I strictly increasing
 * inside every group and within [0, K)) and, if they are malformed, sets a
 * bit of the status word that onexn_device_status reports as ONEXN_EDEVICE.
 * The kernels clamp every P and I they read, so a malformed list faults
 * nothing; the output is then not meaningful.  Costs one small launch. */
#define ONEXN_CHECK_INPUT 0x80u
/* Kernel selection (bits 8..11).  AUTO picks by dtype, N and density:
 * the tensor-core GEMM when its workspace fits and its dense work is
 * estimated to take less time than the FFMA kernel's kept work. */
#define ONEXN_ALGO_SHIFT 8
#define ONEXN_ALGO_MASK (0xFu << ONEXN_ALGO_SHIFT)
#define ONEXN_ALGO_AUTO (0u << ONEXN_ALGO_SHIFT)
#define ONEXN_ALGO_FMA (1u << ONEXN_ALGO_SHIFT)   /* CUDA-core FFMA, any N, fp32/bf16 */
#define ONEXN_ALGO_MMA (2u << ONEXN_ALGO_SHIFT)   /* bf16 sparse tensor-core kernel: each group's
                                                     kept activations gathered into tensor memory,
                                                     one MMA per 16 kept blocks (Eq. 7); N in
                                                     {16, 32, 64, 128}; workspace: its plan */
#define ONEXN_ALGO_TC (3u << ONEXN_ALGO_SHIFT)    /* tcgen05 GEMM on the decoded mask: bf16,
                                                     or fp32 as three tf32 products */

/* Message for the last failed call on this thread ("" if none). */
const char *onexn_last_error(void);

/* Library ABI version, (major << 16) | minor. */
int onexn_version(void);

/*
 * onexn_keep_count -- number of blocks the mask keeps (Eq. 1 constraint
 * ||T||_0 / K = 1 - p).  The rate is taken at a resolution of 1e-6 and
 * keep = round-half-up(total * (1 - p)) in exact int64 arithmetic.
 * EINVAL if rate is outside [0, 1], total < 0 or keep is NULL.
 */
onexn_status onexn_keep_count(int64_t total_blocks, double rate, int64_t *keep);

/*
 * onexn_prune -- the 1xN mask of Eq. 4 / Eq. 5: score every block by its l1
 * norm, keep the top (1 - rate) fraction of blocks (onexn_keep_count).
 *   W      host fp32 OIHW [C_out][C_in][KH][KW], read only.
 *   N      block width; must divide C_out.
 *   rate   pruning rate p in [0, 1].
 *   gran   ONEXN_GRAN_TAP or ONEXN_GRAN_KERNEL.
 *   mask   host uint8 [G][K], written in full (caller-owned).
 *   kept   number of kept blocks at the chosen granularity (so the number
 *          of kept indices is kept, or kept*KH*KW for GRAN_KERNEL).
 * A block's score is the sum of |w| over its weights in fp64, in the order
 * n, then kh, then kw.  Ties go to the lower block index g*nb + b (nb = K
 * for TAP, C_in for KERNEL).  The result is deterministic.
 * EINVAL: NULL pointer, N < 1, N not dividing C_out, non-positive dims,
 * rate outside [0, 1].  ENOMEM: scratch allocation failed.
 */
onexn_status onexn_prune(const float *W, int C_out, int C_in, int KH, int KW, int N,
                         double rate, int gran, uint8_t *mask, int64_t *kept);

/*
 * onexn_rearrange -- filter rearrangement of Sec. 3.3, in place.
 *   W_l    host fp32 OIHW [C_out][C_in][KH][KW]; its filters (output
 *          channels) are re-ordered by l1 norm, largest first; equal norms
 *          keep their original order.
 *   W_next nullable host fp32 OIHW [C_out_next][C_out][KH_next][KW_next];
 *          its input channels get the same permutation, so the composition
 *          of the two layers is unchanged.
 *   perm   host int32 [C_out]: perm[o'] = original index now at o'.  Apply
 *          it to anything else indexed by layer l's outputs (bias, BN,
 *          depthwise channels in between).
 * The norm of filter o is the fp64 sum of |w| in (c, kh, kw) order.
 * EINVAL: NULL W_l/perm, non-positive dims.  ENOMEM: scratch failed.
 */
onexn_status onexn_rearrange(float *W_l, int C_out, int C_in, int KH, int KW,
                             float *W_next, int C_out_next, int KH_next, int KW_next,
                             int32_t *perm);

/*
 * onexn_pack -- BSR encoding of Sec. 3.4 (Fig. 3).
 *   W, mask   as in onexn_prune (host).
 *   wdtype    ONEXN_F32 (D is float) or ONEXN_BF16 (D is bfloat16 bits,
 *             round-to-nearest-even of the fp32 weight).
 *   P         host int32 [G+1]; I host int32 [t_cap]; D host [t_cap][N].
 *   t         out: number of kept blocks t (= sum of mask).
 * Col-group g's kept indices are written in increasing k order into
 * I[P[g] .. P[g+1]), with their N weights in the same rows of D.
 * EINVAL: NULL pointer, bad dims, t_cap smaller than the kept count (t is
 * still written), a mask byte other than 0/1.
 */
onexn_status onexn_pack(const float *W, const uint8_t *mask, int C_out, int C_in, int KH,
                        int KW, int N, int wdtype, int32_t *P, int32_t *I, void *D,
                        int64_t t_cap, int64_t *t);

/*
 * onexn_prune_device -- onexn_prune on the GPU, bit for bit the same mask,
 * for weights that live in device memory (re-pruning inside a fine-tuning
 * loop without a host round trip).
 *   W        DEVICE fp32 OIHW [C_out][C_in][KH][KW].
 *   mask     DEVICE uint8 [G][K], written in full.
 *   kept     HOST out: the kept block count (onexn_keep_count; known
 *            without reading the device).
 *   workspace, workspace_bytes
 *            DEVICE scratch, 256-byte aligned, of at least
 *            onexn_prune_device_workspace_size bytes (the blocks' norms and
 *            the selection state); calls that run concurrently need their
 *            own.
 *   stream   cudaStream_t (NULL = legacy default stream).
 * Scores, order and tie rule as onexn_prune (fp64 l1 norms summed n, kh, kw;
 * larger first, then the lower block index).  Asynchronous; no allocation.
 * EINVAL as onexn_prune, plus a short or misaligned workspace; ECUDA on a
 * launch failure.
 */
onexn_status onexn_prune_device_workspace_size(int C_out, int C_in, int KH, int KW, int N, int gran,
                                               size_t *bytes);
onexn_status onexn_prune_device(const float *W, int C_out, int C_in, int KH, int KW, int N, double rate,
                                int gran, uint8_t *mask, int64_t *kept, void *workspace,
                                size_t workspace_bytes, void *stream);

/*
 * onexn_pack_device -- onexn_pack on the GPU, bit for bit the same P, I, D.
 *   W, mask  DEVICE (as onexn_prune_device); mask bytes are 0 or 1 (any
 *            non-zero byte counts as kept).
 *   wdtype   ONEXN_F32 or ONEXN_BF16 (round-to-nearest-even).
 *   P        DEVICE int32 [G+1], written in full (P[G] = the mask's count).
 *   I, D     DEVICE int32 [t_cap] and [t_cap][N]: the kept blocks at
 *            z < t_cap are written; t_cap must be at least the mask's count
 *            (e.g. onexn_prune_device's kept, times KH*KW for
 *            ONEXN_GRAN_KERNEL), else the blocks past it are left out while
 *            P still counts them.
 *   workspace, workspace_bytes
 *            DEVICE scratch of onexn_pack_device_workspace_size bytes (the
 *            per-group counts).
 * Asynchronous; no allocation.  EINVAL: NULL pointers, bad dims, N not
 * dividing C_out, unknown wdtype, short workspace.  ECUDA on a launch failure.
 */
onexn_status onexn_pack_device_workspace_size(int C_out, int N, size_t *bytes);
onexn_status onexn_pack_device(const float *W, const uint8_t *mask, int C_out, int C_in, int KH, int KW,
                               int N, int wdtype, int32_t *P, int32_t *I, void *D, int64_t t_cap,
                               void *workspace, size_t workspace_bytes, void *stream);

/*
 * onexn_packed_validate -- host check of a BSR index structure before it is
 * copied to the device: P[0] = 0, P non-decreasing, P[G] = t, each
 * col-group's I strictly increasing and inside [0, K).  EINVAL on the first
 * violation (the message names it).
 */
onexn_status onexn_packed_validate(const int32_t *P, const int32_t *I, int G, int64_t t,
                                   int K);

/* Geometry of one convolution.  Output size per dimension:
 * Ho = (H + 2*pad_h - dil_h*(KH-1) - 1) / stride_h + 1 (same for W). */
typedef struct {
    int B, H, W, C_in;                 /* input  x: [B][H][W][C_in]   */
    int C_out, KH, KW;                 /* weights: [C_out][C_in][KH][KW] */
    int stride_h, stride_w;
    int pad_h, pad_w;                  /* zero padding */
    int dil_h, dil_w;
} onexn_conv_desc;

/* Output spatial size of desc; EINVAL if it is empty or desc is invalid. */
onexn_status onexn_conv_out_shape(const onexn_conv_desc *desc, int *Ho, int *Wo);

/*
 * onexn_conv_fwd -- forward convolution of a 1xN-pruned layer, computed
 * block by block from the BSR weights (Eq. 7):
 *   y[p, gN:(g+1)N] = bias[gN:(g+1)N] + sum_{z=P[g]}^{P[g+1]-1} X[p, I[z]] * D[z, :]
 * where X[p, k] is the input value under output pixel p at tap
 * (kh, kw) = ((k / C_in) / KW, (k / C_in) % KW) and channel c = k % C_in
 * (zero in the padding), followed by max(., 0) if flags has ONEXN_RELU.
 *
 *   desc    host pointer to the geometry.
 *   P, I, D DEVICE pointers to the BSR weights of onexn_pack (N, t as
 *           packed; D's element type must equal dtype).  P and I must pass
 *           onexn_packed_validate; the kernels never read outside
 *           I[0..t) and D[0..t*N) even if they do not.
 *   x       DEVICE NHWC activations, fp32 (dtype ONEXN_F32) or bf16
 *           (ONEXN_BF16), 16-byte aligned; C_in % 4 == 0 (fp32) or
 *           C_in % 8 == 0 (bf16).
 *   y       DEVICE NHWC output [B][Ho][Wo][C_out], same element type as x,
 *           16-byte aligned, must not overlap x.  bf16 outputs are the
 *           round-to-nearest-even of the fp32 result.
 *   bias    nullable DEVICE fp32 [C_out].
 *   dtype   ONEXN_F32: fp32 inputs and weights, fp32 accumulation.
 *           ONEXN_BF16: bf16 inputs and weights, fp32 accumulation.
 *   flags   ONEXN_RELU or ONEXN_RELU6, | one ONEXN_ALGO_* value,
 *           | ONEXN_DECODED (weights already decoded in the workspace),
 *           | ONEXN_REUSE_DECODE (AUTO hint: the decode will be reused).
 *   workspace, workspace_bytes
 *           nullable DEVICE scratch owned by the caller, 256-byte aligned.
 *           Some kernel families need it (onexn_conv_workspace_size): the
 *           tensor-core GEMM (ALGO_TC) decodes the weights into it; the
 *           sparse tensor-core kernel (ALGO_MMA) writes its plan there (per
 *           64-channel chunk and tile of 128/N groups: the groups' kept
 *           entry counts and channels and those entries' D rows, 16944
 *           bytes).  The call overwrites
 *           it, so calls that run concurrently need separate workspaces.
 *           AUTO only picks a family whose minimum workspace fits in
 *           workspace_bytes.
 *   stream  cudaStream_t to launch on (NULL = legacy default stream).
 * Asynchronous: returns after the launch; errors of the launch itself are
 * returned as ECUDA.  No allocation, no synchronisation, no host read of
 * device memory.  EINVAL: bad geometry, N not dividing C_out, alignment,
 * NULL pointers, a forced ALGO whose workspace does not fit.
 * EUNSUPPORTED: the forced ALGO cannot run this case.
 */
onexn_status onexn_conv_fwd(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I,
                            const void *D, int N, int64_t t, const void *x, void *y,
                            const float *bias, int dtype, unsigned flags, void *workspace,
                            size_t workspace_bytes, void *stream);

/*
 * onexn_conv_fwd_ex -- onexn_conv_fwd with a residual input:
 *   y = act(conv(x) + bias + residual)
 * (the residual add of MobileNet-V2's inverted-residual block, fused into the
 * convolution's epilogue; the paper's Eq. 7 output plus a skip connection).
 *   residual  nullable DEVICE NHWC [B][Ho][Wo][C_out] of dtype, 16-byte
 *             aligned; it may be y itself (y += conv(x) + bias) but must not
 *             partially overlap y.
 * Everything else as onexn_conv_fwd, which is onexn_conv_fwd_ex with
 * residual = NULL.
 */
onexn_status onexn_conv_fwd_ex(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I,
                               const void *D, int N, int64_t t, const void *x, void *y,
                               const float *bias, const void *residual, int dtype, unsigned flags,
                               void *workspace, size_t workspace_bytes, void *stream);

/*
 * onexn_dwconv_fwd -- the dense depthwise convolution between the pruned
 * expand and project 1x1 convolutions of MobileNet-V2's inverted-residual
 * block (not pruned; no paper equation of its own):
 *   y[b,oh,ow,c] = act(bias[c] + sum_{kh,kw} W[c][kh][kw]
 *                  * x[b, oh*sh - ph + kh*dh, ow*sw - pw + kw*dw, c])
 *   desc    geometry with C_in == C_out == C; C % 4 == 0 (fp32) or % 8 (bf16).
 *   W       DEVICE fp32 [C][KH][KW], 16-byte aligned; bias nullable DEVICE fp32 [C].
 *   x, y    DEVICE NHWC of dtype (ONEXN_F32 / ONEXN_BF16; bf16 outputs are
 *           the RNE of the fp32 result), 16-byte aligned, not overlapping.
 *   flags   0, ONEXN_RELU or ONEXN_RELU6.
 *   stream  cudaStream_t (NULL = legacy default stream).
 * Asynchronous; no allocation.  EINVAL on bad geometry, alignment, NULL
 * pointers or flags; ECUDA on a launch failure.
 */
onexn_status onexn_dwconv_fwd(const onexn_conv_desc *desc, const float *W, const float *bias,
                              const void *x, void *y, int dtype, unsigned flags, void *stream);

/*
 * Fine-tuning with the mask held fixed (the pruned network is fine-tuned
 * after pruning, Sec. 4.1; the pruned blocks stay zero).  desc is the
 * forward geometry: x [B][H][W][C_in], dy [B][Ho][Wo][C_out] = the
 * gradient of the loss with respect to the forward's PRE-activation output
 * (the caller applies the activation's backward, and the residual branch
 * takes dy as it is).  C_out must be a multiple of 8.
 *
 * onexn_conv_bwd_data -- the input gradient
 *   dx[b,ih,iw,c] = sum over (o, kh, kw, oh, ow) with oh*sh - ph + kh*dh = ih
 *                   and ow*sw - pw + kw*dw = iw of W[o,c,kh,kw] * dy[b,oh,ow,o]
 * over the kept blocks (P, I, D as for onexn_conv_fwd).
 *   dy, dx  DEVICE NHWC of dtype, 16-byte aligned, not overlapping; dx is
 *           written in full (or added to, with ONEXN_ACCUMULATE).
 *   flags   0 or ONEXN_ACCUMULATE.
 *   workspace, workspace_bytes
 *           DEVICE scratch of onexn_conv_bwd_data_workspace_size bytes,
 *           256-byte aligned (the decoded weights and their flipped
 *           transpose); concurrent calls need their own.
 * Stride-1 layers run on the tensor-core GEMM (dx is a convolution of dy
 * with the flipped, transposed weights); strided ones on a direct kernel.
 * fp32: three tf32 products per term as the forward; bf16: bf16 products,
 * fp32 accumulation, RNE output.  Asynchronous; no allocation.
 * EINVAL as onexn_conv_fwd plus a short workspace; EUNSUPPORTED: C_out % 8.
 */
onexn_status onexn_conv_bwd_data_workspace_size(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                                                size_t *bytes);
onexn_status onexn_conv_bwd_data(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I,
                                 const void *D, int N, int64_t t, const void *dy, void *dx, int dtype,
                                 unsigned flags, void *workspace, size_t workspace_bytes, void *stream);

/*
 * onexn_conv_bwd_weight -- the gradient of the kept weights, in BSR order:
 *   dD[z][n] = sum_{b,oh,ow} dy[b,oh,ow,gN+n] * x[b, oh*sh - ph + kh*dh,
 *              ow*sw - pw + kw*dw, c]      for P[g] <= z < P[g+1],
 *              I[z] = (kh*KW + kw)*C_in + c
 * (the layout of D, so an optimizer updates D in place), and optionally the
 * bias gradient db[o] = sum dy[..., o].
 *   P, I    DEVICE BSR indices (as packed; D itself is not needed).
 *   x, dy   DEVICE NHWC of dtype, 16-byte aligned.
 *   dD      DEVICE fp32 [t][N]; db nullable DEVICE fp32 [C_out].
 *   workspace, workspace_bytes
 *           DEVICE scratch of onexn_conv_bwd_weight_workspace_size bytes,
 *           256-byte aligned: dy and the im2col view of x transposed to
 *           pixel-contiguous rows (fp32: the latter as tf32 high and low
 *           parts), pixels padded to 64, plus one 128 x BN fp32 partial
 *           tile per GEMM item.
 * The products run on the tensor cores (fp32: three tf32 products per
 * term; bf16: exact bf16 products) with fp32 accumulation over pixel
 * slices, added in slice order (deterministic).  Asynchronous.
 * EINVAL: bad geometry or pointers, short workspace; EUNSUPPORTED: C_out % 8.
 */
onexn_status onexn_conv_bwd_weight_workspace_size(const onexn_conv_desc *desc, int N, int dtype, size_t *bytes);
onexn_status onexn_conv_bwd_weight(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I, int N,
                                   int64_t t, const void *x, const void *dy, float *dD, float *db, int dtype,
                                   void *workspace, size_t workspace_bytes, void *stream);

/*
 * onexn_dwproj_fwd -- MobileNet-V2's depthwise 3x3 + ReLU6 fused into the
 * 1xN-pruned 1x1 projection that follows it (fp32, tensor-core family):
 *   y = act(Proj(relu6(dw(h))) + bias + residual)
 * where dw(h)[b,oh,ow,c] = b_dw[c] + sum_{kh,kw} W_dw[kh*3+kw][c]
 * * h[b, oh*s - 1 + kh, ow*s - 1 + kw, c] (zero padding) and Proj is Eq. 7
 * with (P, I, D) on the depthwise's output grid; the depthwise output is
 * computed inside the GEMM's A operand path and never stored.
 *   dw_desc  the depthwise geometry: B, H, W, C_in = C_out = C, 3x3,
 *            stride 1 or 2 (both dims), pad 1, dilation 1.
 *   W_dw     DEVICE fp32 [9][C], TAP-major (note: onexn_dwconv_fwd takes
 *            [C][3][3]), 16-byte aligned; b_dw nullable DEVICE fp32 [C].
 *   P, I, D, N, t  the projection's BSR weights (C_out x C); C_out % 8 == 0.
 *   h        DEVICE fp32 NHWC [B][H][W][C], 16-byte aligned; y DEVICE fp32
 *            [B][Ho][Wo][C_out], not overlapping h; bias, residual as for
 *            onexn_conv_fwd_ex.
 *   flags    ONEXN_RELU / ONEXN_RELU6 (of the projection), ONEXN_DECODED,
 *            ONEXN_REUSE_DECODE, ONEXN_ALGO_AUTO or ONEXN_ALGO_TC.
 *   workspace  as onexn_conv_fwd for the 1x1 projection with ONEXN_ALGO_TC
 *            (onexn_conv_workspace_size of that layer).
 * Asynchronous; no allocation.  EUNSUPPORTED for bf16 or a projection the
 * tensor-core family cannot run; EINVAL otherwise as onexn_conv_fwd_ex.
 */
onexn_status onexn_dwproj_fwd(const onexn_conv_desc *dw_desc, const float *W_dw, const float *b_dw,
                              const int32_t *P, const int32_t *I, const void *D, int N, int64_t t, int C_out,
                              const void *h, void *y, const float *bias, const void *residual, int dtype,
                              unsigned flags, void *workspace, size_t workspace_bytes, void *stream);

/*
 * onexn_conv_workspace_size -- bytes of device workspace onexn_conv_fwd
 * needs for these arguments with this flags' ALGO (for AUTO: the largest
 * need among the families AUTO may pick, so that passing this many bytes
 * lets AUTO choose freely).  ONEXN_ALGO_TC needs at least the decoded
 * masked weights: C_out * KH*KW*C_in bf16 values (dtype ONEXN_BF16), or
 * twice C_out * KH*KW*C_in fp32 values, their tf32 high and low parts
 * (ONEXN_F32), rounded up to 256 bytes; the size reported here adds the
 * space its GEMM uses to spread the last, partial round of output tiles
 * over all SMs (one 128 x BN fp32 partial tile for each of 152 CTAs, BN =
 * 64, 128 or 256 by C_out, and 152 flags).  With only the minimum the GEMM
 * runs without that balancing.  ONEXN_ALGO_FMA needs none.
 */
onexn_status onexn_conv_workspace_size(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                                       unsigned flags, size_t *bytes);

/*
 * onexn_conv_algo -- which kernel family onexn_conv_fwd would run for these
 * arguments and this much workspace (an ONEXN_ALGO_* value other than
 * AUTO), without launching.  EINVAL / EUNSUPPORTED as onexn_conv_fwd.
 */
onexn_status onexn_conv_algo(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                             unsigned flags, size_t workspace_bytes, unsigned *algo);

/*
 * onexn_conv_tc_form -- which form the tensor-core family's GEMM takes for
 * these arguments (Eq. 6 / Eq. 7 on the decoded weights in every form; they
 * differ in how the activations reach the tensor cores), without launching:
 *   ONEXN_GEMM_IM2COL        one TMA im2col tile of 128 output pixels per
 *                            (tap, 64-channel chunk)
 *   ONEXN_GEMM_IM2COL_WIDE   the same on tiles of 256 output pixels (two
 *                            halves sharing each weight tile; bf16)
 *   ONEXN_GEMM_HALO_RESIDENT stride-1 spatial bf16 layers: tiles of whole
 *                            output rows, one load of the tile's input rows
 *                            per channel chunk read by every tap, the column
 *                            tile's weights kept in shared memory
 *   ONEXN_GEMM_HALO_STREAMED the same input loads on tiles of 256 positions
 *                            of the padded output, weights streamed
 * Reads the current device's SM count (152 when there is no device).
 * EINVAL as onexn_conv_fwd's shape checks.
 */
#define ONEXN_GEMM_IM2COL 0
#define ONEXN_GEMM_IM2COL_WIDE 1
#define ONEXN_GEMM_HALO_RESIDENT 2
#define ONEXN_GEMM_HALO_STREAMED 3
onexn_status onexn_conv_tc_form(const onexn_conv_desc *desc, int N, int64_t t, int dtype, int *form);

/*
 * onexn_conv_halo_geometry -- the plan of the streamed halo form
 * (ONEXN_GEMM_HALO_STREAMED) for a bf16 layer, for inspection and tests;
 * no device work.  The output is laid out in a padded space of Hp rows of
 * Wp positions per image (position (n*Hp + r)*Wp + c is output pixel
 * (n, r, c) when r < Ho and c < Wo).  A strided layer is split into the
 * phases of its input (Eq. 6's taps regrouped by which input pixels they
 * read).  The halo load at padded position (r, c) starts at input base
 * (lower_w + stride_w*c, lower_h + stride_h*r), steps by the strides, and
 * reads x at base + the phase's offsets, zeros outside x.  Tap k of a phase
 * reads the load from row shift(k) on.
 *   geom    HOST int[8]: Wp, Hp, lower_w, lower_h, positions per halo load,
 *           phases, taps, column tile.
 *   taps    HOST uint32[49]: per tap in phase order, (kh*KW + kw) << 16 | shift.
 *   phases  HOST uint32[4]: first tap | end tap << 8 | w offset << 16 |
 *           h offset << 24.
 * Reads the current device's SM count (152 when there is no device).
 * EINVAL as onexn_conv_fwd's shape checks or a NULL output; EUNSUPPORTED
 * when the layer has no streamed plan (1x1, too much padding, ...).  The
 * GEMM may still run another form (onexn_conv_tc_form decides).
 */
onexn_status onexn_conv_halo_geometry(const onexn_conv_desc *desc, int N, int64_t t, int *geom,
                                      uint32_t *taps, uint32_t *phases);

/*
 * onexn_conv_fwd_host -- onexn_conv_fwd on activations in HOST memory:
 * y_host = conv(x_host), with the copies to and from the GPU inside the
 * call.  The batch is cut into chunks of whole images; each chunk is copied
 * in, convolved and copied out on internal streams so that the copy
 * engines and the SMs overlap (the tensor-core family decodes the weights
 * once per call).
 *   desc, P, I, D, N, t, bias, dtype, flags
 *           as onexn_conv_fwd (P, I, D, bias are DEVICE pointers).
 *   x_host  HOST NHWC input [B][H][W][C_in] of dtype.  Pinned memory
 *           (cudaHostAlloc / cudaHostRegister) lets the copies run
 *           asynchronously; pageable memory works but serialises them.
 *   y_host  HOST NHWC output [B][Ho][Wo][C_out] of dtype, same rules.
 *   workspace, workspace_bytes
 *           DEVICE scratch, 256-byte aligned, at least
 *           onexn_conv_host_workspace_size bytes: the decoded weights (if
 *           any) and three device slots each for an input and an output
 *           chunk.  Overwritten; concurrent calls need separate workspaces.
 *   stream  the caller's stream: the call's work starts after the work
 *           enqueued on it before the call, and the stream waits for the
 *           call's last copy, so synchronising it makes y_host valid.
 *           Calls on different streams (with different workspaces) overlap.
 * Asynchronous like onexn_conv_fwd; neither x_host nor y_host may be
 * touched by the host until the stream has been synchronised.  Errors as
 * onexn_conv_fwd, plus EINVAL for a NULL host pointer (B > 0) or a
 * workspace that is too small; an ECUDA in the middle of the enqueueing
 * leaves the chunks already enqueued running.
 */
onexn_status onexn_conv_fwd_host(const onexn_conv_desc *desc, const int32_t *P, const int32_t *I,
                                 const void *D, int N, int64_t t, const void *x_host, void *y_host,
                                 const float *bias, int dtype, unsigned flags, void *workspace,
                                 size_t workspace_bytes, void *stream);

/*
 * onexn_conv_host_workspace_size -- bytes of device workspace
 * onexn_conv_fwd_host needs for these arguments (no GPU needed).
 */
onexn_status onexn_conv_host_workspace_size(const onexn_conv_desc *desc, int N, int64_t t, int dtype,
                                            unsigned flags, size_t *bytes);

/*
 * onexn_conv_fwd_noalloc -- onexn_conv_fwd for callers that cannot allocate
 * device memory.  The paper has no counterpart; it is a deployment aid.
 *
 * It runs the tensor-core family (ONEXN_ALGO_TC; flags may carry
 * ONEXN_RELU and AUTO or TC) with its scratch -- the decoded weight matrix,
 * as sized by onexn_conv_workspace_size -- in a fixed 8 MiB array that is part of
 * the library's device image, instead of a caller workspace.  It never
 * calls cudaMalloc, cudaFree or any other allocating routine.  Who needs it:
 * code running while a stream is captured into a CUDA graph (allocating
 * there breaks the capture), hosts that forbid allocation after start-up to
 * keep latency predictable, and plug-ins that only receive raw pointers
 * from a framework that owns all device memory.
 *   Arguments as onexn_conv_fwd (x, y, P, I, D, bias are caller-owned).
 *   EINVAL: the decoded weights would exceed 8 MiB (use onexn_conv_fwd with
 *   a workspace), or another ALGO was forced.  EUNSUPPORTED: the
 *   tensor-core family cannot run the case (channel counts, strides).
 * Every GPU that loads the library keeps the 8 MiB until the process exits.
 * All calls share the array, so calls that overlap on the GPU (different
 * streams or host threads) race and may return wrong results.  Each call
 * rewrites the part it uses before reading it; nothing needs clearing.  The
 * first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture starts.
 */
onexn_status onexn_conv_fwd_noalloc(const onexn_conv_desc *desc, const int32_t *P,
                                    const int32_t *I, const void *D, int N, int64_t t,
                                    const void *x, void *y, const float *bias, int dtype,
                                    unsigned flags, void *stream);

/*
 * onexn_device_status -- read, and clear if `clear` is non-zero, the status
 * word that the kernels of this library keep on the current device (a
 * 4-byte __device__ variable of the library).  A kernel whose bounded
 * internal wait (about one second) runs out sets it and returns early, so
 * its output is not valid; the checked mode's validation kernel
 * (ONEXN_CHECK_INPUT) sets it when the BSR lists are malformed.
 * Synchronises the device first.
 *   *status = ONEXN_OK (nothing reported since the last clear),
 *             ONEXN_EDEVICE (malformed P / I seen in checked mode) or
 *             ONEXN_ETIMEOUT.
 * ECUDA if a runtime call fails (for instance an earlier kernel fault).
 */
onexn_status onexn_device_status(int clear, int *status);

/*
 * onexn_selftest_timeout -- check the timeout path without a faulted GPU:
 * launches on `stream` a one-thread kernel that waits, with the same bounded
 * wait the library's kernels use, on an mbarrier that nothing signals.  The
 * wait runs out after about one second (2^31 SM cycles) and the kernel sets
 * the status word, so a later onexn_device_status reports ONEXN_ETIMEOUT
 * (clear it there); the context stays usable.  Asynchronous; returns ECUDA
 * only if the launch fails.
 */
onexn_status onexn_selftest_timeout(void *stream);

/*
 * Measurement kernels behind the library's rooflines (no paper counterpart;
 * they compute nothing of the method).  Launch only, on `stream`; the caller
 * times them with CUDA events and derives the rates.
 *
 * onexn_probe_ffma -- `blocks` blocks of 256 threads; every thread runs 8
 * independent fp32 fused multiply-add chains of `iters` steps, i.e.
 * 16 * iters flops per thread.  `sink` (DEVICE, >= blocks floats) is only
 * written if the chains reach an impossible value.  EINVAL on blocks or
 * iters < 1 or a NULL sink.
 */
onexn_status onexn_probe_ffma(int blocks, int iters, float *sink, void *stream);

/*
 * onexn_probe_mma_issue -- one CTA per SM; lane 0 of each of `issuers`
 * (1..8) warps issues 4 * iters back-to-back tcgen05.mma (kind::f16, bf16
 * operands of zero, fp32 accumulate, M = 128, K = 16, width N in {16, 32})
 * into its own accumulator, the A operand read from tensor memory
 * (a_tmem != 0) or from shared memory.  2 * 128 * N * 16 * 4 * iters flops
 * per issuer per SM.  EINVAL on other N / issuers or iters < 1.
 */
onexn_status onexn_probe_mma_issue(int N, int issuers, int a_tmem, int iters, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* ONEXN_H */
