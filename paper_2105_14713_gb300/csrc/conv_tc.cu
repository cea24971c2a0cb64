// bf16 tensor-core (tcgen05) kernel of the 1xN-pruned convolution.
//
// The kept blocks of Eq. 7 are first decoded from (P, I, D) into the masked
// weight matrix W[o][k] (bf16, K-major, zero where a block was pruned),
// Omega-bar of Eq. 6, in a caller-provided workspace: a memset, then one
// thread per kept weight D[z][n] writes it to W[gN + n][I[z]].  The layer output
// Y = X (im2col) * W^T is then an implicit GEMM on the 5th-generation tensor
// cores: per tile M = 128 consecutive output pixels x BN output channels,
// K walked in chunks of one tap x 64 channels.
//
// Warp roles (6 warps, one persistent CTA per SM):
//  * warp 0, producer: one thread issues, per chunk, a TMA im2col load of the
//    A tile (128 output pixels x 64 channels of the tap: the hardware walks
//    the output pixels across rows and images and reads zeros in the
//    padding) and a TMA tiled load of the B tile (BN rows x 64 of W), both
//    in the 128-byte-swizzled K-major layout the tensor core reads, counted
//    in bytes on the stage's "full" mbarrier (ring of S stages).
//  * warp 1, MMA: allocates 2*BN TMEM columns (a double-buffered 128 x BN
//    fp32 accumulator); one thread waits "full", issues four
//    tcgen05.mma (K = 16 each) per chunk and commits them to the stage's
//    "empty" mbarrier; after the last chunk of a tile it commits to the
//    accumulator's "tmem_full" mbarrier.
//  * warps 2-5, epilogue: wait "tmem_full", read the accumulator with
//    tcgen05.ld (warp w reads TMEM lanes 32*(w%4)..+31 = its 32 pixels),
//    release it ("tmem_empty") so the MMA warp can reuse the buffer, add the
//    bias, apply ReLU, round to bf16 into a 128-byte-swizzled staging tile
//    in shared memory, and write the tile to y[p][o] with TMA bulk stores.
// For 1x1, stride-1, unpadded layers the A tile is a plain 2-D box of
// x viewed as [B*H*W][C_in] (tiled TMA) instead of an im2col load.
// All waits are bounded (about one second each); on expiry the status word
// gets ONEXN_ETIMEOUT, every role stops, outstanding MMAs are drained and
// the TMEM is freed before the kernel returns.
#include "conv_common.cuh"
#include "onexn_internal.h"
#include "tc_ptx.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

namespace onexn {

namespace {

constexpr int kProdWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kEpiWarps = 4;          // warps 2..5
constexpr int kThreadsTc = 32 * 6;
constexpr int kBM = 128;              // pixels per tile (UMMA M)
constexpr int kBK = 64;               // channels per chunk: one 128-byte swizzle row

template <int BN>
struct TcLayout {
    static constexpr int kS = BN >= 256 ? 3 : 6;              // stages in the ring
    static constexpr int kA = kBM * kBK * 2;                  // 16 KB
    static constexpr int kB = BN * kBK * 2;                   // 8/16/32 KB
    static constexpr int kStage = kA + kB;                    // multiple of 1024
    static constexpr int kOut = kS * kStage;                  // output staging: BN/64 atoms
    static constexpr int kOutBytes = kBM * BN * 2;            //   of [128 rows][64 cols] bf16
    static constexpr int kBias = kOut + kOutBytes;            // BN fp32
    static constexpr int kBar = kBias + BN * 4;
    // full[S], empty[S], tmem_full[2], tmem_empty[2], drain, then the TMEM holder
    static constexpr int kHolder = kBar + (2 * kS + 5) * 8;
    static constexpr int kBytes = kHolder + 16;
    static constexpr int kAlloc = kBytes + 1024;              // room to align the base to 1024
};

// ---------------------------------------------------------------------------
// Decode of the BSR weights into the masked dense matrix W[o][k] (K-major),
// after W has been zeroed: CTA (x, g) scatters kept weights e = 256x + tid of
// col-group g, i.e. D[z][n] with z = P[g] + e / N, n = e % N, to
// W[g*N + n][I[z]].
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
bsr_scatter_kernel(const int32_t *__restrict__ P, const int32_t *__restrict__ I,
                   const __nv_bfloat16 *__restrict__ D, int N, int t, int K,
                   __nv_bfloat16 *__restrict__ W)
{
    const int g = blockIdx.y;
    const int z0 = clampi(__ldg(P + g), 0, t), z1 = clampi(__ldg(P + g + 1), z0, t);
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (z1 - z0) * N) return;
    const int z = z0 + e / N, n = e - (e / N) * N;
    const int k = __ldg(I + z);
    if (k >= 0 && k < K) W[static_cast<int64_t>(g * N + n) * K + k] = D[static_cast<int64_t>(z) * N + n];
}

// barrier over the 4 epilogue warps that also returns the AND of `ok`
__device__ __forceinline__ bool epi_all(bool ok)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, 1, 128, p;\n\tselp.u32 %0, 1, 0, q;\n\t}\n"
        : "=r"(r)
        : "r"(ok ? 1u : 0u)
        : "memory");
    return r != 0;
}

template <int BN>
__global__ void __launch_bounds__(kThreadsTc, 1)
tc_conv_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_x,
               const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_y,
               const int n_tiles, const int n_tn, const int a_tiled)
{
    using L = TcLayout<BN>;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    const uint32_t bar_full = base + L::kBar;
    const uint32_t bar_empty = bar_full + 8 * L::kS;
    const uint32_t bar_tfull = bar_empty + 8 * L::kS;
    const uint32_t bar_tempty = bar_tfull + 16;
    const uint32_t bar_drain = bar_tempty + 16;
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + L::kHolder);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < L::kS; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar_tfull + 8 * b, 1);
            mbar_init(bar_tempty + 8 * b, 32 * kEpiWarps);
        }
        mbar_init(bar_drain, 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tc::tmem_alloc(smem_u32(holder), 2 * BN);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;

    const int n_cchunk = (a.C + kBK - 1) / kBK;
    const int n_chunks = a.KH * a.KW * n_cchunk;
    const int my_tiles = blockIdx.x < n_tiles ? (n_tiles - 1 - blockIdx.x) / gridDim.x + 1 : 0;
    auto abort_now = [&]() { atomicOr(a.status, kStatusTimeout); };

    if (warp == kProdWarp) {
        // ============================ producer ============================
        if (lane == 0) {
            const int hw = a.Ho * a.Wo;
            int item = 0;
            bool failed = false;
            for (int ti = 0; ti < my_tiles && !failed; ++ti) {
                const int u = blockIdx.x + ti * gridDim.x;
                const int tm = u / n_tn, tn = u - tm * n_tn;
                // first output pixel of the tile -> its traversal start (w, h, n)
                const int p0 = tm * kBM;
                const int b0 = p0 / hw, r0 = p0 - b0 * hw;
                const int oh0 = r0 / a.Wo, ow0 = r0 - oh0 * a.Wo;
                const int w0 = ow0 * a.sw - a.pw, h0 = oh0 * a.sh - a.ph;
                int kh = 0, kw = 0, cc0 = 0, k0tap = 0;
                for (int c = 0; c < n_chunks; ++c, ++item) {
                    const int st = item % L::kS;
                    if (item >= L::kS &&
                        !mbar_wait(bar_empty + 8 * st, ((item / L::kS) + 1) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    const uint32_t sa = base + st * L::kStage, sb = sa + L::kA;
                    tc::mbar_arrive_expect_tx(bar_full + 8 * st, L::kStage);
                    if (a_tiled)
                        tc::tma_load_2d(sa, &tmap_x, cc0, p0, bar_full + 8 * st);
                    else
                        tc::tma_load_im2col_4d(sa, &tmap_x, cc0, w0, h0, b0,
                                               static_cast<uint16_t>(kw * a.dw), static_cast<uint16_t>(kh * a.dh),
                                               bar_full + 8 * st);
                    tc::tma_load_2d(sb, &tmap_w, k0tap + cc0, tn * BN, bar_full + 8 * st);
                    cc0 += kBK;
                    if (cc0 >= a.C) {
                        cc0 = 0; k0tap += a.C;
                        if (++kw == a.KW) { kw = 0; ++kh; }
                    }
                }
            }
        }
        __syncwarp();
    } else if (warp == kMmaWarp) {
        // ============================== MMA ==============================
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, BN);
            int item = 0;
            bool failed = false;
            for (int ti = 0; ti < my_tiles && !failed; ++ti) {
                const int acc = ti & 1;
                if (ti >= 2 && !mbar_wait(bar_tempty + 8 * acc, ((ti >> 1) + 1) & 1)) {
                    abort_now(); failed = true; break;
                }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + acc * BN;
                for (int c = 0; c < n_chunks; ++c, ++item) {
                    const int st = item % L::kS;
                    if (!mbar_wait(bar_full + 8 * st, (item / L::kS) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    tc::fence_after_sync();
                    const uint32_t sa = base + st * L::kStage, sb = sa + L::kA;
                    const uint64_t ad = tc::desc_kmajor_sw128(sa), bd = tc::desc_kmajor_sw128(sb);
#pragma unroll
                    for (int kk = 0; kk < kBK / 16; ++kk)
                        tc::mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, (c | kk) != 0);
                    tc::commit(bar_empty + 8 * st);
                }
                if (!failed) tc::commit(bar_tfull + 8 * acc);
            }
            // Drain: everything this thread issued has completed before the TMEM is freed.
            tc::commit(bar_drain);
            if (!mbar_wait(bar_drain, 0)) abort_now();
        }
        __syncwarp();
    } else {
        // ============================ epilogue ============================
        const int q = warp & 3;                      // TMEM lanes 32q .. 32q+31
        const int row = 32 * q + lane;               // pixel row of the tile
        const bool leader = (warp == kMmaWarp + 1) && lane == 0;
        float *sbias = reinterpret_cast<float *>(smem + L::kBias);
        const uint32_t sout = base + L::kOut;
        for (int ti = 0; ti < my_tiles; ++ti) {
            const int acc = ti & 1;
            // all four warps take the same decision (tcgen05.ld and the named
            // barriers below need all of them)
            if (!epi_all(mbar_wait(bar_tfull + 8 * acc, (ti >> 1) & 1))) { abort_now(); break; }
            tc::fence_after_sync();
            const int u = blockIdx.x + ti * gridDim.x;
            const int tm = u / n_tn, tn = u - tm * n_tn;
            // the staging tile is free once the previous tile's stores have read it
            if (leader) tc::bulk_wait_read0();
            for (int c = row; c < BN; c += 128) {
                const int o = tn * BN + c;
                sbias[c] = (a.bias && o < a.C_out) ? __ldg(a.bias + o) : 0.f;
            }
            tc::named_bar(1, 128);
            // read the accumulator in batches of up to 128 columns (registers)
            constexpr int kGrp = BN < 128 ? BN : 128;
#pragma unroll
            for (int g0 = 0; g0 < BN; g0 += kGrp) {
                uint32_t r[kGrp / 32][32];
#pragma unroll
                for (int cb = 0; cb < kGrp / 32; ++cb)
                    tc::ld_32x32b_x32(tmem + (static_cast<uint32_t>(32 * q) << 16) + acc * BN + g0 + 32 * cb,
                                      r[cb]);
                tc::ld_wait();
                if (g0 + kGrp >= BN) {
                    tc::fence_before_sync();
                    mbar_arrive(bar_tempty + 8 * acc);   // accumulator free for tile ti + 2
                }
#pragma unroll
                for (int cb = 0; cb < kGrp / 32; ++cb) {
#pragma unroll
                    for (int v8 = 0; v8 < 4; ++v8) {
                        const int c = g0 + 32 * cb + 8 * v8;  // first of 8 columns
                        float f[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            float val = __uint_as_float(r[cb][8 * v8 + e]) + sbias[c + e];
                            if (a.relu) val = fmaxf(val, 0.f);
                            f[e] = val;
                        }
                        const int atom = c >> 6, jj = (c & 63) >> 3;
                        const uint32_t dst = sout + atom * (kBM * 128) + row * 128 + ((jj ^ (row & 7)) << 4);
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(dst),
                                     "r"(pack_bf16x2(f[0], f[1])), "r"(pack_bf16x2(f[2], f[3])),
                                     "r"(pack_bf16x2(f[4], f[5])), "r"(pack_bf16x2(f[6], f[7]))
                                     : "memory");
                    }
                }
            }
            tc::fence_proxy_async_smem();
            tc::named_bar(1, 128);
            if (leader) {
#pragma unroll
                for (int at = 0; at < BN / 64; ++at)
                    if (tn * BN + 64 * at < a.C_out)
                        tc::tma_store_2d(&tmap_y, tn * BN + 64 * at, tm * kBM, sout + at * (kBM * 128));
                tc::bulk_commit();
            }
        }
        if (leader) tc::bulk_wait0();
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 2 * BN);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_tiled_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

PFN_cuTensorMapEncodeIm2col_v12000 encode_im2col_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeIm2col_v12000 fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeIm2col_v12000>(p);
    });
    return fn;
}

// Bounding box of the im2col traversal (innermost spatial dim first: W, H):
// window start positions run from -pad to dim - 1 + pad - dil*(k-1).
void im2col_corners(const ConvArgs &a, int lower[2], int upper[2])
{
    lower[0] = -a.pw;
    lower[1] = -a.ph;
    upper[0] = a.pw - a.dw * (a.KW - 1);
    upper[1] = a.ph - a.dh * (a.KH - 1);
}

// 2-D bf16 tensor map over a row-major [rows][cols] matrix, box 64 x box_rows,
// 128-byte swizzle, zero fill outside.
bool tmap_2d(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows)
{
    auto enc_t = encode_tiled_fn();
    if (!enc_t) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return enc_t(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                 CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN>
cudaError_t launch_bn(const ConvArgs &a, const __nv_bfloat16 *W, cudaStream_t st)
{
    using L = TcLayout<BN>;
    auto kern = tc_conv_kernel<BN>;
    const int K = a.KH * a.KW * a.C;
    auto enc_i = encode_im2col_fn();
    if (!enc_i) return cudaErrorNotSupported;
    // A: a 1x1, stride-1, unpadded layer reads x as a [B*H*W][C] matrix; any
    // other layer reads x[B][H][W][C] as an im2col view (128 pixels x 64
    // channels per load).
    const int a_tiled = (a.KH == 1 && a.KW == 1 && a.sh == 1 && a.sw == 1 && a.ph == 0 && a.pw == 0);
    CUtensorMap tmap_x;
    if (a_tiled) {
        if (!tmap_2d(&tmap_x, a.x, static_cast<uint64_t>(a.B) * a.H * a.W, a.C, kBM)) return cudaErrorInvalidValue;
    } else {
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(a.C), static_cast<cuuint64_t>(a.W),
                                    static_cast<cuuint64_t>(a.H), static_cast<cuuint64_t>(a.B)};
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(a.C) * 2,
                                       static_cast<cuuint64_t>(a.C) * 2 * a.W,
                                       static_cast<cuuint64_t>(a.C) * 2 * a.W * a.H};
        int lower[2], upper[2];
        im2col_corners(a, lower, upper);
        const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(a.sw), static_cast<cuuint32_t>(a.sh), 1};
        if (enc_i(&tmap_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(a.x), dims, strides,
                  lower, upper, kBK, kBM, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    // B: W[C_out][K] bf16, box 64 (K) x BN rows.  y: [P_pix][C_out] bf16,
    // stored in boxes of 64 columns x 128 rows (rows/columns outside y are
    // not written).
    CUtensorMap tmap_w, tmap_y;
    if (!tmap_2d(&tmap_w, W, a.C_out, K, BN)) return cudaErrorInvalidValue;
    if (!tmap_2d(&tmap_y, a.y, a.P_pix, a.C_out, kBM)) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc);
    if (e != cudaSuccess) return e;
    int sms = 0;
    e = device_sm_count(&sms);
    if (e != cudaSuccess) return e;
    const int n_tm = (a.P_pix + kBM - 1) / kBM;
    const int n_tn = (a.C_out + BN - 1) / BN;
    const int n_tiles = n_tm * n_tn;
    const int grid = n_tiles < sms ? n_tiles : sms;
    kern<<<grid, kThreadsTc, L::kAlloc, st>>>(a, tmap_x, tmap_w, tmap_y, n_tiles, n_tn, a_tiled);
    return cudaGetLastError();
}

}  // namespace

size_t tc_workspace_bytes(const ConvArgs &a)
{
    const size_t bytes = static_cast<size_t>(a.C_out) * a.KH * a.KW * a.C * 2;
    return (bytes + 255) & ~static_cast<size_t>(255);
}

// bf16 inputs; C_in, C_out multiples of 8 (16-byte rows); the im2col box
// corners within the TMA's [-128, 127] range; strides <= 8; 16-bit offsets.
bool tc_supports(const ConvArgs &a)
{
    if (a.C % 8 || a.C_out % 8) return false;
    if (a.sh > 8 || a.sw > 8) return false;
    int lower[2], upper[2];
    im2col_corners(a, lower, upper);
    for (int i = 0; i < 2; ++i)
        if (lower[i] < -128 || lower[i] > 127 || upper[i] < -128 || upper[i] > 127) return false;
    if ((a.KH - 1) * a.dh > 65535 || (a.KW - 1) * a.dw > 65535) return false;
    return true;
}

cudaError_t launch_tc(const ConvArgs &a, void *workspace, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    __nv_bfloat16 *W = static_cast<__nv_bfloat16 *>(workspace);
    const int K = a.KH * a.KW * a.C;
    cudaError_t e = cudaMemsetAsync(W, 0, static_cast<size_t>(a.C_out) * K * 2, st);
    if (e != cudaSuccess) return e;
    if (a.t > 0) {
        const int64_t per_group = static_cast<int64_t>(K) * a.N;     // upper bound of t_g * N
        const dim3 grid(static_cast<unsigned>((per_group + 255) / 256), a.C_out / a.N);
        bsr_scatter_kernel<<<grid, 256, 0, st>>>(a.P, a.I, static_cast<const __nv_bfloat16 *>(a.D), a.N, a.t,
                                                 K, W);
        e = cudaGetLastError();
    }
    if (e != cudaSuccess) return e;
    if (a.C_out <= 64) return launch_bn<64>(a, W, st);
    if (a.C_out <= 128) return launch_bn<128>(a, W, st);
    return launch_bn<256>(a, W, st);
}

}  // namespace onexn
