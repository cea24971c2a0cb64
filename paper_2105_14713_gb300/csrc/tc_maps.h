// TMA descriptors of the activation operand shared by the tensor-core
// kernels (conv_tc.cu, conv_mma.cu).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>

#include "conv_common.cuh"

namespace onexn {

// 1 when x is read as a plain [B*H*W][C] matrix (1x1, stride 1, no padding).
int tc_x_tiled(const ConvArgs &a);
// Encode (or fetch from the cache) the tensor map of x: boxes of 128 output
// pixels x bk channels (128 bytes), 128-byte swizzle; false on failure.
bool tc_x_tmap(const ConvArgs &a, CUtensorMapDataType type, int elem, int bk, CUtensorMap *tmap_x);
// The driver's im2col tensor-map encoder (nullptr if unavailable).
PFN_cuTensorMapEncodeIm2col_v12000 encode_im2col_fn_public();
// Encode (or fetch) a tiled tensor map of rank 2..4, 128-byte swizzle, zero
// fill: dims and box innermost first, strides[i] = byte stride of dim i + 1.
bool tc_tmap_tiled(CUtensorMap *m, CUtensorMapDataType type, int rank, const void *ptr, const uint64_t *dims,
                   const uint64_t *strides, const uint32_t *box);

}  // namespace onexn
