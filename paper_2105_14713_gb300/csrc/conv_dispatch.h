// Argument checks, kernel-family selection and launches shared by the
// convolution entry points (conv_fwd.cu, conv_host.cu, conv_noalloc.cu).
#pragma once

#include <cuda_runtime.h>

#include "conv_common.cuh"
#include "onexn.h"

namespace onexn {

cudaError_t launch_fma(const ConvArgs &a, int dtype, cudaStream_t st);
// sparse tensor-core family (bf16): a plan of the kept lists (per chunk and
// group tile: entry counts, channels and D rows) in the workspace
// (mma_workspace_bytes), then the kernel
cudaError_t launch_mma(const ConvArgs &a, void *workspace, size_t ws_bytes, cudaStream_t st);
bool mma_supports(const ConvArgs &a);
size_t mma_workspace_bytes(const ConvArgs &a);
// tensor-core family: decode of (P, I, D) into the workspace, then the GEMM
// (which splits its last round of tiles across CTAs when ws_bytes has room
// for tc_workspace_bytes, else needs tc_workspace_min)
cudaError_t launch_tc(const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes, cudaStream_t st);
cudaError_t tc_decode(const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes, cudaStream_t st);
cudaError_t tc_gemm(const ConvArgs &a, int dtype, const void *workspace, size_t ws_bytes, cudaStream_t st);
bool tc_supports(const ConvArgs &a, int dtype);
size_t tc_workspace_bytes(const ConvArgs &a, int dtype);
size_t tc_workspace_min(const ConvArgs &a, int dtype);
// AUTO's time estimate of the tensor-core family (ns; fixed costs relative to FFMA's)
double tc_cost_ns(const ConvArgs &a, int dtype, size_t ws_bytes, bool decoded);
// The tensor-core GEMM on caller-given operands (backward passes).
cudaError_t tc_gemm_weights(const ConvArgs &a, int dtype, const void *W, const void *W_lo, void *sk_space,
                            cudaStream_t st);
struct TcSplitPlan {
    int bn, tiles, n_tn, split_s;
    size_t partial_bytes;
};
TcSplitPlan tc_split_plan(int M, int Ncols, int64_t K, int dtype);
cudaError_t tc_gemm_split(const ConvArgs &a, int dtype, const void *W, const void *W_lo, float *partials,
                          const TcSplitPlan &plan, cudaStream_t st);
size_t tc_weights_bytes(const ConvArgs &a, int dtype);
// Forms of the tensor-core GEMM (values of onexn_conv_tc_form).
enum : int { kGemmIm2col = 0, kGemmIm2colWide = 1, kGemmHaloResident = 2, kGemmHaloStreamed = 3 };
// Halo-tile forms of the bf16 GEMM for stride-1 spatial layers (conv_halo.cu):
// which one takes the layer (against the im2col GEMM's column tile;
// kGemmIm2col for none), and the launch on the decoded weights W[C_out][K].
int halo_form(const ConvArgs &a, int im2col_bn);
cudaError_t halo_gemm(const ConvArgs &a, const void *W, int im2col_bn, cudaStream_t st);
// The form the tensor-core GEMM takes for this layer and dtype (conv_tc.cu).
int tc_gemm_form(const ConvArgs &a, int dtype);
// The streamed halo form's plan geometry (conv_halo.cu): geom[8], taps[49],
// phases[4]; false when the layer has no streamed plan.
bool halo_streamed_geometry(const ConvArgs &a, int geom[8], uint32_t *taps, uint32_t *phases);
size_t tc_sk_bytes(const ConvArgs &a, int dtype);

namespace detail {

// Shape, dtype and flag checks; fills the geometry part of *a.
onexn_status check_shape(const onexn_conv_desc *d, int N, int64_t t, int dtype, unsigned flags,
                         ConvArgs *a);
// Device-pointer checks; fills the pointer part of *a.
onexn_status check_pointers(const int32_t *P, const int32_t *I, const void *D, const void *x,
                            void *y, const float *bias, int dtype, ConvArgs *a);
// Workspace a family uses at best / needs at least for these arguments.
size_t workspace_for(unsigned algo, const ConvArgs &a, int dtype);
size_t workspace_min_for(unsigned algo, const ConvArgs &a, int dtype);
// Can the family run this case at all (dtype, shape)?
bool supports(unsigned algo, const ConvArgs &a, int dtype);
// The family onexn_conv_fwd runs (flags' forced ALGO, else the AUTO choice).
unsigned pick_algo(const ConvArgs &a, int dtype, unsigned flags, size_t ws_bytes);
onexn_status check_algo(unsigned algo, const ConvArgs &a, int dtype, size_t ws_bytes);
// Launch one family (decode included for the tensor-core family).
cudaError_t launch(unsigned algo, const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes,
                   cudaStream_t st);
// Checked mode: the device-side validation of (P, I) (status bit on failure).
cudaError_t launch_validate(const ConvArgs &a, cudaStream_t st);

}  // namespace detail
}  // namespace onexn
