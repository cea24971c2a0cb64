// Tensor-core (tcgen05) kernels of the 1xN-pruned convolution.
//
// The kept blocks of Eq. 7 are first decoded from (P, I, D) into the masked
// weight matrix W[o][k] (K-major, zero where a block was pruned), Omega-bar
// of Eq. 6, in a caller-provided workspace, by one kernel that writes every
// element once.  The layer output
// Y = X (im2col) * W^T is then an implicit GEMM on the 5th-generation tensor
// cores: per tile M = 128 consecutive output pixels x BN output channels,
// K walked in chunks of one tap x 128 bytes of channels (64 bf16 / 32 fp32).
//
// Two element types share the kernel:
//  * bf16 inputs: one tcgen05.mma.kind::f16 per K step of 16, fp32 accumulate.
//  * fp32 inputs: each product is split into tf32 parts,
//      x*w ~= x_hi*w_hi + x_lo*w_hi + x_hi*w_lo,
//    three tcgen05.mma.kind::tf32 per K step of 8 into one fp32 accumulator.
//    w_hi = w rounded to tf32 and w_lo = w - w_hi are decoded into the
//    workspace; x_hi = x with its 13 low mantissa bits cleared and
//    x_lo = x - x_hi are computed per chunk from the A tile in shared memory
//    and written to tensor memory, from where the MMAs read A (so shared
//    memory only feeds them B).  Both hi parts are exact tf32 values, so the
//    products do not depend on how the tensor core reduces an fp32 operand
//    to tf32.  The dropped x_lo*w_lo term and the tf32 reduction of the lo
//    parts are ~2^-20 relative to |x*w|.
//
// Warp roles (one persistent CTA per SM):
//  * warp 0, producer: one thread issues, per chunk, a TMA im2col load of the
//    A tile (128 output pixels x 128 bytes of channels of the tap: the
//    hardware walks the output pixels across rows and images and reads zeros
//    in the padding; for 1x1, stride-1, unpadded layers a plain tiled 2-D box
//    of x viewed as [B*H*W][C_in]) and tiled TMA loads of the B tile(s)
//    (BN rows x 128 bytes of W), all in the 128-byte-swizzled K-major layout
//    the tensor core reads, counted in bytes on the stage's "full" mbarrier.
//  * warps 6-9 (fp32 only), split: wait "full" (and for the TMEM A slot to
//    be free: "empty" of the chunk two back), read one pixel row of the A
//    tile each, write x_hi | x_lo to the slot's TMEM lanes, arrive "split".
//  * warp 1, MMA: allocates the TMEM (a double-buffered 128 x BN fp32
//    accumulator, plus the A ring for fp32); one thread waits for the stage ("full", or "split"
//    for fp32), issues the MMAs of the chunk and commits them to the
//    stage's "empty" mbarrier; after the last chunk of a tile it commits to
//    the accumulator's "tmem_full" mbarrier.
//  * warps 2-5, epilogue: wait "tmem_full", read the accumulator with
//    tcgen05.ld (warp w reads TMEM lanes 32*(w%4)..+31 = its 32 pixels),
//    release it ("tmem_empty"), add the bias, apply ReLU and store NHWC one
//    128-byte column atom at a time through a double-buffered
//    128-byte-swizzled staging tile and TMA stores.
// All waits are bounded (about one second each); on expiry the status word
// gets ONEXN_ETIMEOUT, every role stops, outstanding MMAs are drained and
// the TMEM is freed before the kernel returns.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "onexn_internal.h"
#include "tc_ptx.cuh"
#include "tc_maps.h"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <type_traits>
#include <cstring>
#include <mutex>

namespace onexn {

namespace {

constexpr int kProdWarp = 0;
constexpr int kMmaWarp = 1;
constexpr int kEpiWarp0 = 2;          // warps 2..5 (fp32), 2..9 (bf16)
constexpr int kSplitWarp0 = 6;        // warps 6..9 (fp32 only)
constexpr int kBM = 128;              // pixels per tile (UMMA M)
constexpr int kRowBytes = 128;        // bytes of K per tile row: one 128-byte swizzle row

struct TcBf16 {
    using T = __nv_bfloat16;
    static constexpr bool kSplit = false;
    static constexpr int kBK = 64;                 // channels per chunk
    static constexpr int kKStep = 16;              // K per MMA
    static constexpr CUtensorMapDataType kTmap = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    // warps: producer, MMA, and eight epilogue warps, two per TMEM lane
    // quarter taking every other 64-column atom: an epilogue warp is bound
    // by its own latencies (~0.5 us per 128 x 64 atom), so a second warp per
    // quarter doubles the output rate of tiles with short K loops
    static constexpr int kWarps = 10;
    static constexpr int kEpiWarps = 8;
    static constexpr int kMT = 1;                  // 128-row halves per tile
};
// bf16 with 256-row tiles: the two 128-row halves have their own
// accumulators and A tiles and share every B tile, so a K chunk moves
// 2 x 16 KB of A and one B tile for twice the multiply-adds
struct TcBf16W : TcBf16 {
    static constexpr int kMT = 2;
};
struct TcF32 {
    using T = float;
    static constexpr bool kSplit = true;
    static constexpr int kBK = 32;
    static constexpr int kKStep = 8;
    static constexpr CUtensorMapDataType kTmap = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    static constexpr int kWarps = 10;              // warps 6-9 split x into tf32 parts
    static constexpr int kEpiWarps = 4;
    static constexpr int kMT = 1;
};

constexpr int kSmemMax = 232448;      // dynamic shared memory per CTA (opt-in maximum)
constexpr int kAccMax = 4;            // accumulator buffers in TMEM at most
constexpr int kPlanCTAs = 152;        // stream-K: partial slots / flags for at most this many CTAs
                                      // (GB300's SM count; a larger GPU splits over 152 of its SMs)
constexpr int kMinSplitIters = 4;     // stream-K: at least this many chunk iterations per CTA

// Stream-K moves partial tiles through global memory and makes a finisher
// wait for them; on GB300 that pays only when a tile's own K loop is long:
// from 16 chunks per tile for fp32 (three tf32 MMAs per chunk) and 32 for
// bf16, measured on batch-1 MobileNet-V2 and ResNet-50 layers; 256-row bf16
// tiles do twice the work per chunk and are fewer, from 8 chunks.
constexpr int sk_min_chunks(bool split, int MT = 1) { return split ? 16 : (MT > 1 ? 8 : 32); }

// one partial slot (128 MT x BN fp32) per CTA
constexpr size_t sk_partial_bytes(int BN, int MT = 1) { return static_cast<size_t>(kPlanCTAs) * kBM * MT * BN * 4; }

constexpr int pow2_at_least(int v, int p = 32) { return p >= v ? p : pow2_at_least(v, 2 * p); }

template <typename Tr, int BN>
struct TcLayout {
    static constexpr int kA = Tr::kMT * kBM * kRowBytes;             // 16 KB per 128-row half
    static constexpr int kB = BN * kRowBytes;                        // 8/16/32 KB
    static constexpr int kStage = kA + (Tr::kSplit ? 2 * kB : kB);   // [A | B_hi | B_lo]
    static constexpr int kTx = kStage;                               // bytes the TMA brings
    // output staging: per epilogue warp buffers of 32 rows x one 128-byte
    // column atom, two per warp with four epilogue warps, one with eight
    static constexpr int kOutBufs = Tr::kEpiWarps == 4 ? 2 : 1;
    static constexpr int kOutBytes = Tr::kEpiWarps * kOutBufs * 32 * kRowBytes;
    static constexpr int kFixed = 1024 + kOutBytes + BN * 4 + (3 * 6 + 2 * 4 + 2) * 8 + 16;
    static constexpr int kS = ((kSmemMax - kFixed) / kStage) > 6 ? 6 : ((kSmemMax - kFixed) / kStage);
    static constexpr int kOut = kS * kStage;
    static constexpr int kBias = kOut + kOutBytes;                   // BN fp32
    static constexpr int kBar = kBias + BN * 4;
    // full[S], split[S], empty[S], tmem_full[4], tmem_empty[4], drain, fixup, TMEM holder
    static constexpr int kHolder = kBar + (3 * kS + 2 * kAccMax + 2) * 8;
    static constexpr int kBytes = kHolder + 16;
    static constexpr int kAlloc = kBytes + 1024;                      // room to align the base to 1024
    // TMEM columns: the fp32 accumulator buffers (two when they fit next to
    // the A ring, else one) and, for the split form, a ring of two A slots
    // of 64 columns (x_hi in the first 32, x_lo in the next 32).
    static constexpr int kARing = Tr::kSplit ? 128 : 0;
    // as many accumulator buffers as fit next to the A ring (up to 4): the
    // MMA of tile i + kAcc waits for the epilogue of tile i, so layers with
    // few chunks per tile need several to keep the tensor core busy
    static constexpr int kAccCols = Tr::kMT * BN;                   // one accumulator: both halves
    static constexpr int kAccFit = (512 - kARing) / kAccCols;
    static constexpr int kAcc = kAccFit > kAccMax ? kAccMax : kAccFit;
    static constexpr int kTmemCols = pow2_at_least(kAcc * kAccCols + kARing);
    // a stream-K tile has at most kMaxParts parts besides the finisher's (as
    // many 128 x BN fp32 tiles as the stage ring's bytes), which bounds the
    // additions in the finisher's epilogue
    static constexpr int kSlotBytes = Tr::kMT * kBM * BN * 4;
    // 256-row tiles: the finisher reads its parts from L2 atom by atom, so
    // their number is not bound by the stage ring; four keep the split fine
    static constexpr int kMaxParts = Tr::kMT > 1 ? 4 : kS * kStage / kSlotBytes;
    static_assert(kS >= 2, "ring too small");
    static_assert(kMaxParts >= 1, "stream-K parts");
    static_assert(kAlloc <= kSmemMax, "shared memory");
    static_assert(kTmemCols <= 512, "tensor memory");
};

// ---------------------------------------------------------------------------
// Decode of the BSR weights into the masked dense matrix W[o][k] (K-major).
// CTA (x, g, r) writes the 256 columns k0 = 256x .. k0+255 of rows
// 8r .. 8r+7 (those below N) of col-group g: it marks in shared memory which kept block z of the group
// (if any) sits at each column, then writes every element of the band once,
// coalesced: W[g*N + n][k] = D[z][n] for a kept column, 0 otherwise.  For
// fp32 W gets the tf32 rounding of the value and W_lo the rest.
// ---------------------------------------------------------------------------
constexpr int kDecodeCols = 256;
constexpr int kDecodeRows = 8;

__device__ __forceinline__ float tf32_rna(float v)
{
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;\n" : "=r"(r) : "f"(v));
    return __uint_as_float(r);
}

template <typename T>
__global__ void __launch_bounds__(kDecodeCols)
bsr_decode_kernel(const int32_t *__restrict__ P, const int32_t *__restrict__ I, const T *__restrict__ D,
                  int N, int t, int K, T *__restrict__ W, T *__restrict__ W_lo, int *__restrict__ flags,
                  int n_flags)
{
    __shared__ int32_t zmap[kDecodeCols];
    const int g = blockIdx.y, tid = threadIdx.x;
    // let the GEMM launch and run its prologue meanwhile; it waits for this
    // grid's completion before reading anything
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    // the GEMM's stream-K flags start each launch lowered
    if (flags && (blockIdx.x | blockIdx.y | blockIdx.z) == 0)
        for (int i = tid; i < n_flags; i += kDecodeCols) flags[i] = 0;
    const int k0 = blockIdx.x * kDecodeCols;
    zmap[tid] = -1;
    __syncthreads();
    const int z0 = clampi(__ldg(P + g), 0, t), z1 = clampi(__ldg(P + g + 1), z0, t);
    for (int z = z0 + tid; z < z1; z += kDecodeCols) {
        const int k = __ldg(I + z) - k0;
        if (k >= 0 && k < kDecodeCols) zmap[k] = z;
    }
    __syncthreads();
    const int k = k0 + tid;
    if (k >= K) return;
    const int z = zmap[tid];
    const int n1 = min(N, static_cast<int>(blockIdx.z + 1) * kDecodeRows);
    for (int n = blockIdx.z * kDecodeRows; n < n1; ++n) {
        const int64_t dst = static_cast<int64_t>(g * N + n) * K + k;
        const T v = z >= 0 ? D[static_cast<int64_t>(z) * N + n] : T(0.f);
        if constexpr (sizeof(T) == 4) {
            const float hi = tf32_rna(v);
            W[dst] = hi;
            W_lo[dst] = v - hi;
        } else {
            W[dst] = v;
        }
    }
}

// barrier over the epilogue warps (n threads) that also returns the AND of `ok`
__device__ __forceinline__ bool epi_all(bool ok, int n)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, 1, %2, p;\n\tselp.u32 %0, 1, 0, q;\n\t}\n"
        : "=r"(r)
        : "r"(ok ? 1u : 0u), "r"(n)
        : "memory");
    return r != 0;
}

// Work schedule of one launch, the same in every role of every CTA.  Tiles
// [0, dp_tiles) are whole tiles taken round-robin (CTA b: b, b+G, ...).  The
// chunk iterations of the remaining sk_tiles tiles are cut into sk_ctas
// contiguous ranges, one for each of CTAs 0 .. sk_ctas-1 (stream-K).  A CTA
// runs its stream-K range before its whole tiles, walking it from the end:
// first the start of one tile, then whole tiles, last the end of another.
// A tile cut between CTAs is finished by the highest of them: the others
// (lower CTAs, for which that tile's piece is the first segment they run)
// each write their part to their own partial slot and raise their flag; the
// finisher waits for those flags and adds the parts, read from L2, to its
// own accumulator in CTA order, so the result does not depend on timing.
// The finisher's wait and additions run in its epilogue warps while its MMA
// warp goes on with the whole tiles.  Waiting only on lower CTAs, which
// were scheduled first, cannot deadlock.
//
// Split mode (split_s > 0; plain GEMMs with a long K, e.g. the weight
// gradient whose K is the pixels): item i = slice * n_tiles + tile covers
// chunks [slice * C / S, (slice + 1) * C / S) of its tile; CTA b takes
// items b, b + G, ...; every item's accumulator goes to partial slot i and
// a separate kernel adds the S slots of a tile in slice order.
struct TcSched {
    int n_tiles, n_tn, n_chunks;
    int dp_tiles, sk_tiles, sk_ctas;
    int split_s;
    // every tile of a CTA multiplies the same B (one column tile, or a grid
    // that is a multiple of their number) and its K loop fits in the stage
    // ring: chunk c's B is loaded once into stage c's B region and stays
    // there; the stages then carry A only
    int b_resident;
    // divisors of the per-tile / per-segment index arithmetic
    FastDiv div_tn, div_hw, div_wo, div_cchunk, div_kw;
    float *partials;     // slot b: CTA b's part of a split tile, [BN/4][128] float4
    int *flags;          // [kPlanCTAs]: slot b written
};

struct TcSeg {
    int tile, c0, c1;    // chunk iterations [c0, c1) of tile
    int slot;            // split mode: the item's partial slot
};

__device__ __forceinline__ int64_t sk_start(int b, int64_t W, int G) { return static_cast<int64_t>(b) * W / G; }
// the CTA whose stream-K range holds iteration q (largest b with sk_start(b) <= q)
__device__ __forceinline__ int sk_owner(int64_t q, int64_t W, int G)
{
    return static_cast<int>(((q + 1) * G + W - 1) / W) - 1;
}

struct TcSegIter {
    int b, G, n_dp, i_dp, C, dp_tiles, split_s, n_tiles;
    int64_t s, e;        // stream-K range still to walk: [s, e), from e down
    __device__ TcSegIter(const TcSched &sc)
    {
        b = blockIdx.x;
        G = gridDim.x;
        C = sc.n_chunks;
        dp_tiles = sc.dp_tiles;
        split_s = sc.split_s;
        n_tiles = sc.n_tiles;
        const int items = split_s > 0 ? n_tiles * split_s : dp_tiles;
        n_dp = items > b ? (items - 1 - b) / G + 1 : 0;
        i_dp = 0;
        const int64_t W = static_cast<int64_t>(sc.sk_tiles) * C;
        s = b < sc.sk_ctas ? sk_start(b, W, sc.sk_ctas) : 0;
        e = b < sc.sk_ctas ? sk_start(b + 1, W, sc.sk_ctas) : 0;
    }
    __device__ bool next(TcSeg &sg)
    {
        if (split_s > 0) {
            if (i_dp >= n_dp) return false;
            const int i = b + i_dp * G;
            const int slice = i / n_tiles;
            sg.tile = i - slice * n_tiles;
            sg.c0 = static_cast<int>(static_cast<int64_t>(slice) * C / split_s);
            sg.c1 = static_cast<int>(static_cast<int64_t>(slice + 1) * C / split_s);
            sg.slot = i;
            ++i_dp;
            return true;
        }
        sg.slot = -1;
        // the stream-K pieces first (so that a finisher's fixup overlaps the
        // whole tiles' MMAs instead of trailing the kernel), from the range's
        // end down: the piece a CTA contributes to a tile finished by a
        // higher CTA is always the first segment it runs
        if (e > s) {
            const int t = static_cast<int>((e - 1) / C);
            const int64_t t0 = static_cast<int64_t>(t) * C;
            sg.tile = dp_tiles + t;
            sg.c1 = static_cast<int>(e - t0);
            sg.c0 = s > t0 ? static_cast<int>(s - t0) : 0;
            e -= sg.c1 - sg.c0;
            return true;
        }
        if (i_dp >= n_dp) return false;
        sg.tile = b + i_dp * G;
        sg.c0 = 0;
        sg.c1 = C;
        ++i_dp;
        return true;
    }
};

template <typename Tr, int BN>
__global__ void __launch_bounds__(Tr::kWarps * 32, 1)
tc_conv_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_x,
               const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_wlo,
               const __grid_constant__ CUtensorMap tmap_y, const TcSched sched, const int a_tiled)
{
    using L = TcLayout<Tr, BN>;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    const uint32_t bar_full = base + L::kBar;
    const uint32_t bar_split = bar_full + 8 * L::kS;
    const uint32_t bar_empty = bar_split + 8 * L::kS;
    const uint32_t bar_tfull = bar_empty + 8 * L::kS;
    const uint32_t bar_tempty = bar_tfull + 8 * kAccMax;
    const uint32_t bar_drain = bar_tempty + 8 * kAccMax;
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + L::kHolder);
    // the MMA waits on "split" (fp32: x_hi / x_lo in TMEM) or "full" (bf16)
    const uint32_t bar_ready = Tr::kSplit ? bar_split : bar_full;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < L::kS; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_split + 8 * s, 128);
            mbar_init(bar_empty + 8 * s, 1);
        }
        for (int b = 0; b < kAccMax; ++b) {
            mbar_init(bar_tfull + 8 * b, 1);
            mbar_init(bar_tempty + 8 * b, 32 * Tr::kEpiWarps);
        }
        mbar_init(bar_drain, 1);
        fence_mbar_init();
    }
    if (warp == kMmaWarp) {
        tc::tmem_alloc(smem_u32(holder), L::kTmemCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;
    // Launched as a programmatic dependent of the previous kernel on the
    // stream (the weight decode, or the layer before): everything above
    // overlapped it; global memory is touched only after it (and everything
    // before it on the stream) has completed.  The next kernel may then
    // start its own prologue (it waits the same way before reading).
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

    const int n_cchunk = (a.C + Tr::kBK - 1) / Tr::kBK;
    const int n_tn = sched.n_tn;
    auto abort_now = [&]() { atomicOr(a.status, kStatusTimeout); };
    const bool dw_mode = Tr::kSplit && a.dw_x != nullptr;   // A from the fused depthwise

    if (warp == kProdWarp) {
        // ============================ producer ============================
        if (lane == 0) {
            const int hw = a.Ho * a.Wo;
            int item = 0;
            bool failed = false;
            TcSegIter it(sched);
            TcSeg sg;
            while (!failed && it.next(sg)) {
                const int tm = static_cast<int>(sched.div_tn.div(sg.tile)), tn = sg.tile - tm * n_tn;
                // first output pixel of each 128-row half -> its traversal start (w, h, n)
                const int p0 = tm * (kBM * Tr::kMT);
                int hw0[Tr::kMT], hh0[Tr::kMT], hb0[Tr::kMT];
#pragma unroll
                for (int hf = 0; hf < Tr::kMT; ++hf) {
                    const int ph = p0 + hf * kBM;
                    const int b0 = static_cast<int>(sched.div_hw.div(ph)), r0 = ph - b0 * hw;
                    const int oh0 = static_cast<int>(sched.div_wo.div(r0)), ow0 = r0 - oh0 * a.Wo;
                    hw0[hf] = ow0 * a.sw - a.pw;
                    hh0[hf] = oh0 * a.sh - a.ph;
                    hb0[hf] = b0;
                }
                // chunk c0 -> tap (kh, kw) and channel offset
                const int tap = static_cast<int>(sched.div_cchunk.div(sg.c0));
                int cc0 = (sg.c0 - tap * n_cchunk) * Tr::kBK, k0tap = tap * a.C;
                int kh = static_cast<int>(sched.div_kw.div(tap)), kw = tap - kh * a.KW;
                for (int c = sg.c0; c < sg.c1; ++c, ++item) {
                    const int st = item % L::kS;
                    if (item >= L::kS &&
                        !mbar_wait(bar_empty + 8 * st, ((item / L::kS) + 1) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    const uint32_t sa = base + st * L::kStage;
                    const uint32_t sb = sa + L::kA;
                    // B bytes of this chunk: when B is resident only the CTA's
                    // first tile loads it, chunk c into stage c's B region
                    const bool load_b = !sched.b_resident || item < sched.n_chunks;
                    const uint32_t b_tx = load_b ? static_cast<uint32_t>(L::kTx - L::kA) : 0u;
                    if (dw_mode) {
                        // A comes from the split warps' depthwise; only B is loaded
                        tc::mbar_arrive_expect_tx(bar_full + 8 * st, b_tx);
                    } else {
                        tc::mbar_arrive_expect_tx(bar_full + 8 * st, L::kA + b_tx);
#pragma unroll
                        for (int hf = 0; hf < Tr::kMT; ++hf) {
                            const uint32_t dst = sa + hf * (kBM * kRowBytes);
                            if (a_tiled)
                                tc::tma_load_2d(dst, &tmap_x, cc0, p0 + hf * kBM, bar_full + 8 * st);
                            else
                                tc::tma_load_im2col_4d(dst, &tmap_x, cc0, hw0[hf], hh0[hf], hb0[hf],
                                                       static_cast<uint16_t>(kw * a.dw),
                                                       static_cast<uint16_t>(kh * a.dh), bar_full + 8 * st);
                        }
                    }
                    if (load_b) {
                        tc::tma_load_2d(sb, &tmap_w, k0tap + cc0, tn * BN, bar_full + 8 * st);
                        if constexpr (Tr::kSplit)
                            tc::tma_load_2d(sb + L::kB, &tmap_wlo, k0tap + cc0, tn * BN, bar_full + 8 * st);
                    }
                    cc0 += Tr::kBK;
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
            int item = 0, si = 0;
            bool failed = false;
            TcSegIter it(sched);
            TcSeg sg;
            for (; !failed && it.next(sg); ++si) {
                const int acc = si % L::kAcc, use = si / L::kAcc;
                if (use >= 1 && !mbar_wait(bar_tempty + 8 * acc, (use - 1) & 1)) {
                    abort_now(); failed = true; break;
                }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + acc * L::kAccCols;   // half hf at d_tmem + hf * BN
                for (int c = sg.c0; c < sg.c1; ++c, ++item) {
                    const int st = item % L::kS;
                    if (!mbar_wait(bar_ready + 8 * st, (item / L::kS) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    tc::fence_after_sync();
                    const uint32_t sa = base + st * L::kStage;
                    // this chunk's B: the stage's, or resident in stage c's B region
                    const uint32_t sbm = (sched.b_resident ? base + c * L::kStage : sa) + L::kA;
                    const uint64_t bd = tc::desc_kmajor_sw128(sbm);
                    const uint32_t first = (c == sg.c0) ? 1u : 0u;   // the first chunk overwrites D
                    if constexpr (Tr::kSplit) {
                        constexpr uint32_t idesc = tc::idesc_tf32_f32(kBM, BN);
                        const uint64_t bld = tc::desc_kmajor_sw128(sbm + L::kB);
                        // A slot of this chunk: x_hi columns, then x_lo 32 columns on
                        const uint32_t a_hi = tmem + L::kAcc * L::kAccCols + (item & 1) * 64;
#pragma unroll
                        for (int kk = 0; kk < Tr::kBK / Tr::kKStep; ++kk) {
                            tc::mma_tf32_ta(d_tmem, a_hi + 8 * kk, bd + 2 * kk, idesc, !(first && kk == 0));
                            tc::mma_tf32_ta(d_tmem, a_hi + 32 + 8 * kk, bd + 2 * kk, idesc, 1);
                            tc::mma_tf32_ta(d_tmem, a_hi + 8 * kk, bld + 2 * kk, idesc, 1);
                        }
                    } else {
                        constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, BN);
                        const uint64_t ad = tc::desc_kmajor_sw128(sa);
                        constexpr uint32_t kHalfDesc = kBM * kRowBytes / 16;   // next half's A tile
#pragma unroll
                        for (int kk = 0; kk < Tr::kBK / Tr::kKStep; ++kk)
#pragma unroll
                            for (int hf = 0; hf < Tr::kMT; ++hf)
                                tc::mma_bf16(d_tmem + hf * BN, ad + hf * kHalfDesc + 2 * kk, bd + 2 * kk, idesc,
                                             !(first && kk == 0));
                    }
                    tc::commit(bar_empty + 8 * st);
                }
                if (!failed) tc::commit(bar_tfull + 8 * acc);
            }
            // Drain: everything this thread issued has completed before the TMEM is freed.
            tc::commit(bar_drain);
            if (!mbar_wait(bar_drain, 0)) abort_now();
        }
        __syncwarp();
    } else if (Tr::kSplit && warp >= kSplitWarp0) {
        // ============================ split (fp32) ========================
        // Thread i of warp w owns pixel row 32*(w%4) + i of the tile: it reads
        // the row's 32 fp32 values from the swizzled A tile (logical 16-byte
        // chunk j of row r sits at physical chunk j ^ (r % 8), so the eight
        // rows of a quarter-warp hit eight distinct bank groups), splits them
        // into x_hi = x with the low 13 mantissa bits cleared and
        // x_lo = x - x_hi, and writes both to its TMEM lane in the chunk's A
        // slot (item % 2).  Before overwriting a slot it waits until the MMAs
        // of the chunk two back, which read it, have completed.
        if constexpr (Tr::kSplit) {
            const int q = warp & 3;
            const int row = 32 * q + lane;
            const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * q) << 16) + L::kAcc * L::kAccCols;
            const int hw = a.Ho * a.Wo;
            int64_t item = 0;
            bool failed = false;
            TcSegIter it(sched);
            TcSeg sg;
            while (!failed && it.next(sg)) {
                // dw mode: this thread's output pixel of the tile
                int pb = -1, poh = 0, pow_ = 0;
                if (dw_mode) {
                    const int tm = static_cast<int>(sched.div_tn.div(sg.tile));
                    const int p = tm * kBM * Tr::kMT + row;
                    if (p < a.P_pix) {
                        pb = static_cast<int>(sched.div_hw.div(p));
                        const int r = p - pb * hw;
                        poh = static_cast<int>(sched.div_wo.div(r));
                        pow_ = r - poh * a.Wo;
                    }
                }
                for (int c = sg.c0; c < sg.c1; ++c, ++item) {
                    const int st = static_cast<int>(item % L::kS);
                    if (item >= 2 && !mbar_wait(bar_empty + 8 * static_cast<int>((item - 2) % L::kS),
                                                static_cast<int>((item - 2) / L::kS) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    uint32_t hi[32], lo[32];
                    if (dw_mode) {
                        // the depthwise 3x3 + bias + ReLU6 of channels cb .. cb+31
                        const int cb = c * Tr::kBK;
                        float v[32];
#pragma unroll
                        for (int j = 0; j < 32; ++j) v[j] = 0.f;
                        if (pb >= 0) {
                            const bool full = cb + 32 <= a.C;
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                if (a.dw_b && (full || cb + j < a.C)) v[j] = __ldg(a.dw_b + cb + j);
                            for (int kh = 0; kh < 3; ++kh) {
                                const int ih = poh * a.dw_s - 1 + kh;
                                if (ih < 0 || ih >= a.dw_H) continue;
                                for (int kw = 0; kw < 3; ++kw) {
                                    const int iw = pow_ * a.dw_s - 1 + kw;
                                    if (iw < 0 || iw >= a.dw_W) continue;
                                    const float *xs = a.dw_x + ((static_cast<int64_t>(pb) * a.dw_H + ih) * a.dw_W + iw) *
                                                                   a.C + cb;
                                    const float *ws = a.dw_w + (kh * 3 + kw) * a.C + cb;
#pragma unroll
                                    for (int j4 = 0; j4 < 8; ++j4) {
                                        if (!full && cb + 4 * j4 >= a.C) break;     // C % 4 == 0
                                        const float4 xv = __ldg(reinterpret_cast<const float4 *>(xs) + j4);
                                        const float4 wv = __ldg(reinterpret_cast<const float4 *>(ws) + j4);
                                        v[4 * j4] = fmaf(wv.x, xv.x, v[4 * j4]);
                                        v[4 * j4 + 1] = fmaf(wv.y, xv.y, v[4 * j4 + 1]);
                                        v[4 * j4 + 2] = fmaf(wv.z, xv.z, v[4 * j4 + 2]);
                                        v[4 * j4 + 3] = fmaf(wv.w, xv.w, v[4 * j4 + 3]);
                                    }
                                }
                            }
#pragma unroll
                            for (int j = 0; j < 32; ++j)
                                v[j] = (full || cb + j < a.C) ? fminf(fmaxf(v[j], 0.f), 6.f) : 0.f;
                        }
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            hi[j] = __float_as_uint(v[j]) & 0xffffe000u;
                            lo[j] = __float_as_uint(v[j] - __uint_as_float(hi[j]));
                        }
                        // B of this chunk must have landed before the MMA is released
                        if (!mbar_wait(bar_full + 8 * st, static_cast<int>(item / L::kS) & 1)) {
                            abort_now(); failed = true; break;
                        }
                    } else {
                        if (!mbar_wait(bar_full + 8 * st, static_cast<int>(item / L::kS) & 1)) {
                            abort_now(); failed = true; break;
                        }
                        tc::fence_after_sync();
                        const uint32_t src = base + st * L::kStage + row * kRowBytes;
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            uint32_t vv[4];
                            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];\n"
                                         : "=r"(vv[0]), "=r"(vv[1]), "=r"(vv[2]), "=r"(vv[3])
                                         : "r"(src + ((j ^ (row & 7)) << 4))
                                         : "memory");
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                hi[4 * j + e] = vv[e] & 0xffffe000u;
                                lo[4 * j + e] = __float_as_uint(__uint_as_float(vv[e]) - __uint_as_float(hi[4 * j + e]));
                            }
                        }
                    }
                    const uint32_t slot = lane_base + static_cast<uint32_t>(item & 1) * 64;
                    tc::st_32x32b_x32(slot, hi);
                    tc::st_32x32b_x32(slot + 32, lo);
                    tc::st_wait();
                    tc::fence_before_sync();
                    mbar_arrive(bar_split + 8 * st);
                }
            }
        }
    } else {
        // ============================ epilogue ============================
        // Per tile, column atom by column atom (128 bytes of output columns:
        // 64 bf16 / 32 fp32): read the atom's accumulator columns from TMEM
        // (warp w owns TMEM lanes = pixel rows 32*(w%4)..+31), add the bias
        // (and the residual), apply the activation, convert, write the row
        // into the warp's 128-byte-swizzled staging buffer (two, alternating)
        // and store the warp's 32 x atom box with TMA.  The residual and the
        // activation are compile-time variants chosen once per launch, so the
        // per-value work has no branches (a per-chunk test for the residual
        // alone cost a third of the epilogue on epilogue-bound 1x1 layers).
      auto epilogue = [&](auto res_c, auto act_c) {
        constexpr bool kRes = decltype(res_c)::value;
        constexpr int kAct = decltype(act_c)::value;
        using T = typename Tr::T;
        constexpr int kAtomCols = kRowBytes / static_cast<int>(sizeof(T));
        constexpr int kAtoms = BN / kAtomCols;
        // atoms of the whole accumulator: half hf's atoms follow half hf-1's
        // in the TMEM columns (half hf at column hf * BN), so atom `at` of
        // the accumulator is columns at * kAtomCols .. + kAtomCols - 1
        constexpr int kGA = kAtoms * Tr::kMT;
        constexpr int kLd = kAtomCols / 32;               // tcgen05.ld x32 per atom
        constexpr int kSlotF4 = BN / 4 * kBM * Tr::kMT;  // float4 per partial slot
        const int q = warp & 3;                      // TMEM lanes 32q .. 32q+31
        const int row = 32 * q + lane;               // pixel row of the tile
        const bool leader = (warp == kEpiWarp0) && lane == 0;
        // eight epilogue warps: warp group eg (of nG) takes atoms eg, eg + nG, ...
        constexpr int kEpiThreads = 32 * Tr::kEpiWarps;
        constexpr int nG = Tr::kEpiWarps / 4;
        const int ew = warp - kEpiWarp0;             // this warp among the epilogue warps
        const int eg = ew / 4;
        const int et = 32 * ew + lane;               // this thread among the epilogue threads
        const uint32_t sout = base + L::kOut;
        float *sbias = reinterpret_cast<float *>(smem + L::kBias);
        const int64_t W_sk = static_cast<int64_t>(sched.sk_tiles) * sched.n_chunks;
        int n_emit = 0;                              // atoms stored so far (staging buffer parity)
        int staged_tn = -1;                          // column tile whose bias is in shared memory
        TcSegIter it(sched);
        TcSeg sg;
        for (int si = 0; it.next(sg); ++si) {
            const int acc = si % L::kAcc;
            // all epilogue warps take the same decision (tcgen05.ld and the
            // named barriers below need all of them)
            if (!epi_all(mbar_wait(bar_tfull + 8 * acc, (si / L::kAcc) & 1), kEpiThreads)) { abort_now(); break; }
            tc::fence_after_sync();
            const int tm = static_cast<int>(sched.div_tn.div(sg.tile)), tn = sg.tile - tm * n_tn;
            const uint32_t t_acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + acc * L::kAccCols;
            // read the accumulator columns of atom `at`; release the TMEM after the last
            auto issue_atom = [&](int at, uint32_t (&r)[kLd][32]) {
#pragma unroll
                for (int l = 0; l < kLd; ++l) tc::ld_32x32b_x32(t_acc + at * kAtomCols + 32 * l, r[l]);
            };
            auto release_acc = [&]() {
                tc::fence_before_sync();
                mbar_arrive(bar_tempty + 8 * acc);       // accumulator free for segment si + kAcc
            };
            // four epilogue warps: the atoms in order, the TMEM loads of atom
            // at+1 in flight while atom at is processed; eight: each warp its
            // own atoms (every nG-th), the other warp of its lane quarter
            // covering its latencies.  A warp releases the accumulator as
            // soon as its last columns are in registers (at once if it has
            // none).
            auto run_atoms = [&](auto &&body) {
                if constexpr (nG == 1) {
                    uint32_t r[2][kLd][32];
                    issue_atom(0, r[0]);
                    tc::ld_wait();
                    if (kGA == 1) release_acc();
#pragma unroll
                    for (int at = 0; at < kGA; ++at) {
                        if (at + 1 < kGA) issue_atom(at + 1, r[(at + 1) & 1]);
                        body(at, r[at & 1]);
                        if (at + 1 < kGA) {
                            tc::ld_wait();
                            if (at + 2 == kGA) release_acc();
                        }
                    }
                } else {
                    if (eg >= kGA) release_acc();
#pragma unroll
                    for (int i = 0; i < (kGA + nG - 1) / nG; ++i) {
                        const int at = i * nG + eg;
                        if (at < kGA) {
                            uint32_t r[kLd][32];
                            issue_atom(at, r);
                            tc::ld_wait();
                            if (at + nG >= kGA) release_acc();
                            body(at, r);
                        }
                    }
                }
            };
            // a lower CTA's part: accumulator atoms -> global slot, no pipelining needed
            auto load_atom = [&](int at, uint32_t (&r)[kLd][32]) {
                issue_atom(at, r);
                tc::ld_wait();
                if (at + nG >= kGA) release_acc();
            };
            // bias / ReLU / convert the row's atom values f and store the
            // warp's 32 rows of the atom: each warp has its own two staging
            // buffers (32 rows x 128 bytes) and TMA stores, so no warp waits
            // for another
            // the tile's bias in shared memory, read as broadcast float4
            const float4 *sb4 = reinterpret_cast<const float4 *>(sbias);
            // (only when the column tile changes: consecutive tiles of a
            // CTA often share it, and the global load is a full memory
            // latency on the epilogue's critical path)
            auto stage_bias = [&]() {
                if (tn == staged_tn) return;         // uniform across the epilogue warps
                staged_tn = tn;
                tc::named_bar(1, kEpiThreads);       // the previous tile's reads are done
                for (int c = et; c < BN; c += kEpiThreads) {
                    const int o = tn * BN + c;
                    sbias[c] = (a.bias && o < a.C_out) ? __ldg(a.bias + o) : 0.f;
                }
                tc::named_bar(1, kEpiThreads);
            };
            auto emit_atom = [&](int ga, float (&f)[kAtomCols]) {
                const int at = ga % kAtoms;                           // atom within the half
                const int row0 = (tm * Tr::kMT + ga / kAtoms) * kBM;  // first pixel row of the half
                const int col0 = tn * BN + at * kAtomCols;
                if (col0 >= a.C_out) {               // the whole atom lies past y's columns: no work,
                    ++n_emit;                        // but an (empty) commit group keeps the count
                    if (lane == 0) tc::bulk_commit();
                    return;
                }
                // this warp's staging buffers alternate across its atoms and
                // tiles (two with four epilogue warps); the store that last
                // used the buffer has read it
                const int buf = L::kOutBufs == 2 ? (n_emit & 1) : 0;
                ++n_emit;
                if (lane == 0) {
                    if constexpr (L::kOutBufs == 2) tc::bulk_wait_read1();
                    else tc::bulk_wait_read0();
                }
                __syncwarp();
                const uint32_t wbuf = sout + (ew * L::kOutBufs + buf) * (32 * kRowBytes);
                // the residual row of this atom (16-byte chunks inside y only)
                const uint4 *res = nullptr;
                if constexpr (kRes) {
                    const int pix = row0 + row;
                    if (pix < a.P_pix)
                        res = reinterpret_cast<const uint4 *>(static_cast<const T *>(a.residual) +
                                                              static_cast<int64_t>(pix) * a.C_out + col0);
                }
#pragma unroll
                for (int j = 0; j < 8; ++j) {        // 16-byte chunk j of the row
                    uint32_t w[4];
                    uint32_t rw[4] = {0u, 0u, 0u, 0u};
                    if constexpr (kRes) {
                        if (res && col0 + j * (16 / static_cast<int>(sizeof(T))) < a.C_out) {
                            const uint4 rv = __ldg(res + j);
                            rw[0] = rv.x; rw[1] = rv.y; rw[2] = rv.z; rw[3] = rv.w;
                        }
                    }
                    if constexpr (sizeof(T) == 4) {
                        const float4 bv = sb4[at * (kAtomCols / 4) + j];
                        const float bb[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            float v = f[4 * j + e] + bb[e];
                            if constexpr (kRes) v += __uint_as_float(rw[e]);
                            w[e] = __float_as_uint(activate_c<kAct>(v));
                        }
                    } else {
                        const float4 b0 = sb4[at * (kAtomCols / 4) + 2 * j], b1 = sb4[at * (kAtomCols / 4) + 2 * j + 1];
                        const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            float v0 = f[8 * j + 2 * e] + bb[2 * e], v1 = f[8 * j + 2 * e + 1] + bb[2 * e + 1];
                            if constexpr (kRes) {
                                v0 += bf16lo(rw[e]);
                                v1 += bf16hi(rw[e]);
                            }
                            w[e] = pack_bf16x2(activate_c<kAct>(v0), activate_c<kAct>(v1));
                        }
                    }
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(
                                     wbuf + lane * kRowBytes + ((j ^ (lane & 7)) << 4)),
                                 "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                                 : "memory");
                }
                tc::fence_proxy_async_smem();
                __syncwarp();
                // one commit group per atom (empty for an atom past C_out,
                // above), so that "at most one group pending" always means
                // buf is free
                if (lane == 0) {
                    tc::tma_store_2d(&tmap_y, col0, row0 + 32 * q, wbuf);
                    tc::bulk_commit();
                }
            };

            if (sched.split_s > 0) {
                // ---- split mode: the item's accumulator -> its partial slot ----
                float4 *mine = reinterpret_cast<float4 *>(sched.partials) + static_cast<int64_t>(sg.slot) * kSlotF4;
                if (eg >= kGA) release_acc();
#pragma unroll 1
                for (int at = eg; at < kGA; at += nG) {
                    uint32_t r[kLd][32];
                    load_atom(at, r);
#pragma unroll
                    for (int v4 = 0; v4 < kAtomCols / 4; ++v4) {
                        const int e = 4 * v4;
                        __stcg(mine + (at * kAtomCols / 4 + v4) * kBM + row,
                               make_float4(__uint_as_float(r[e / 32][e % 32]), __uint_as_float(r[e / 32][e % 32 + 1]),
                                           __uint_as_float(r[e / 32][e % 32 + 2]),
                                           __uint_as_float(r[e / 32][e % 32 + 3])));
                    }
                }
                continue;
            }
            if (sg.c0 == 0 && sg.c1 == sched.n_chunks) {
                // ---- whole tile: accumulator -> bias / ReLU -> y ----
                stage_bias();
                run_atoms([&](int at, uint32_t (&r)[kLd][32]) {
                    float f[kAtomCols];
#pragma unroll
                    for (int e = 0; e < kAtomCols; ++e) f[e] = __uint_as_float(r[e / 32][e % 32]);
                    emit_atom(at, f);
                });
                continue;
            }

            // ---- part of a split tile ----
            const int t_sk = sg.tile - sched.dp_tiles;
            const int64_t q0 = static_cast<int64_t>(t_sk) * sched.n_chunks;
            const int b_first = sk_owner(q0, W_sk, sched.sk_ctas);
            const int b_last = sk_owner(q0 + sched.n_chunks - 1, W_sk, sched.sk_ctas);
            if (static_cast<int>(blockIdx.x) != b_last) {
                // a lower CTA: accumulator -> own partial slot, then the flag
                float4 *mine = reinterpret_cast<float4 *>(sched.partials) + static_cast<int64_t>(blockIdx.x) * kSlotF4;
                if (eg >= kGA) release_acc();
#pragma unroll 1
                for (int at = eg; at < kGA; at += nG) {
                    uint32_t r[kLd][32];
                    load_atom(at, r);
#pragma unroll
                    for (int v4 = 0; v4 < kAtomCols / 4; ++v4) {
                        const int e = 4 * v4;
                        __stcg(mine + (at * kAtomCols / 4 + v4) * kBM + row,
                               make_float4(__uint_as_float(r[e / 32][e % 32]), __uint_as_float(r[e / 32][e % 32 + 1]),
                                           __uint_as_float(r[e / 32][e % 32 + 2]),
                                           __uint_as_float(r[e / 32][e % 32 + 3])));
                    }
                }
                __threadfence();
                tc::fence_proxy_async_global();      // the finisher reads the slot with TMA
                tc::named_bar(1, kEpiThreads);
                if (leader) tc::st_release_gpu(sched.flags + blockIdx.x, 1);
                continue;
            }
            // The finisher: wait for the lower CTAs' flags, then add their
            // parts, read from L2, to the accumulator in CTA order.
            const int n_contrib = b_last - b_first;
            bool ok = true;
            if (leader) {
                for (int k = b_first; k < b_last && ok; ++k) {
                    const long long t0 = clock64();
                    while (tc::ld_acquire_gpu(sched.flags + k) == 0)
                        if (clock64() - t0 > (1ll << 31)) { ok = false; break; }
                }
            }
            if (!epi_all(ok, kEpiThreads)) { abort_now(); break; }
            stage_bias();
            const float4 *parts = reinterpret_cast<const float4 *>(sched.partials) +
                                  static_cast<int64_t>(b_first) * kSlotF4;
            run_atoms([&](int at, uint32_t (&r)[kLd][32]) {
                float f[kAtomCols];
#pragma unroll
                for (int e = 0; e < kAtomCols; ++e) f[e] = __uint_as_float(r[e / 32][e % 32]);
                for (int k = 0; k < n_contrib; ++k) {
                    const float4 *part = parts + static_cast<int64_t>(k) * kSlotF4;
                    float4 v[kAtomCols / 4];
#pragma unroll
                    for (int v4 = 0; v4 < kAtomCols / 4; ++v4) v[v4] = __ldcg(part + (at * kAtomCols / 4 + v4) * kBM + row);
#pragma unroll
                    for (int v4 = 0; v4 < kAtomCols / 4; ++v4) {
                        f[4 * v4] += v[v4].x; f[4 * v4 + 1] += v[v4].y; f[4 * v4 + 2] += v[v4].z; f[4 * v4 + 3] += v[v4].w;
                    }
                }
                emit_atom(at, f);
            });
            tc::named_bar(1, kEpiThreads);           // every part has been read
            if (leader)
                for (int k = b_first; k < b_last; ++k) sched.flags[k] = 0;   // ready for the next launch
        }
        if (lane == 0) tc::bulk_wait0();
      };
        if (a.residual) {
            if (a.relu == 2) epilogue(std::true_type{}, std::integral_constant<int, 2>{});
            else if (a.relu == 1) epilogue(std::true_type{}, std::integral_constant<int, 1>{});
            else epilogue(std::true_type{}, std::integral_constant<int, 0>{});
        } else {
            if (a.relu == 2) epilogue(std::false_type{}, std::integral_constant<int, 2>{});
            else if (a.relu == 1) epilogue(std::false_type{}, std::integral_constant<int, 1>{});
            else epilogue(std::false_type{}, std::integral_constant<int, 0>{});
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, L::kTmemCols);
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

// Encoded tensor maps are cached by their encoding inputs (a layer called
// again on the same buffers skips the driver call): a 64-entry direct-mapped
// table keyed by the device and every argument of the encode.
struct TmapKey {
    uint32_t kind, type;
    int32_t dev, pad0;
    uint64_t ptr;
    uint64_t dims[4], strides[3];
    int32_t lower[2], upper[2];
    uint32_t box[4], estr[4];
};

struct TmapEntry {
    bool valid;
    TmapKey key;
    CUtensorMap map;
};

std::mutex g_tmap_mu;
TmapEntry g_tmap_cache[64];

template <typename Encode>
bool tmap_cached(TmapKey &k, CUtensorMap *out, Encode &&encode)
{
    if (cudaGetDevice(&k.dev) != cudaSuccess) return false;
    uint64_t h = 1469598103934665603ull;                      // FNV-1a over the key bytes
    const unsigned char *kb = reinterpret_cast<const unsigned char *>(&k);
    for (size_t i = 0; i < sizeof(TmapKey); ++i) h = (h ^ kb[i]) * 1099511628211ull;
    TmapEntry &e = g_tmap_cache[h & 63];
    {
        std::lock_guard<std::mutex> lk(g_tmap_mu);
        if (e.valid && std::memcmp(&e.key, &k, sizeof(TmapKey)) == 0) {
            *out = e.map;
            return true;
        }
    }
    if (!encode(out)) return false;
    std::lock_guard<std::mutex> lk(g_tmap_mu);
    e.valid = true;
    e.key = k;
    e.map = *out;
    return true;
}

// 2-D tensor map over a row-major [rows][cols] matrix of `elem`-byte values,
// box 128 bytes x box_rows, 128-byte swizzle, zero fill outside.
bool tmap_2d(CUtensorMap *m, CUtensorMapDataType type, int elem, const void *ptr, uint64_t rows,
             uint64_t cols, uint32_t box_rows)
{
    auto enc_t = encode_tiled_fn();
    if (!enc_t) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * elem};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kRowBytes / elem), box_rows};
    const cuuint32_t estr[2] = {1, 1};
    TmapKey k;
    std::memset(&k, 0, sizeof k);
    k.kind = 0;
    k.type = static_cast<uint32_t>(type);
    k.ptr = reinterpret_cast<uint64_t>(ptr);
    k.dims[0] = cols; k.dims[1] = rows;
    k.strides[0] = strides[0];
    k.box[0] = box[0]; k.box[1] = box[1];
    return tmap_cached(k, m, [&](CUtensorMap *mm) {
        return enc_t(mm, type, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    });
}

}  // namespace

PFN_cuTensorMapEncodeIm2col_v12000 encode_im2col_fn_public() { return encode_im2col_fn(); }

// Tiled tensor map of rank 2..4 with the 128-byte swizzle and zero fill
// outside the tensor, cached like the others.  dims / box innermost first;
// strides[i] is the byte stride of dimension i + 1.
bool tc_tmap_tiled(CUtensorMap *m, CUtensorMapDataType type, int rank, const void *ptr, const uint64_t *dims,
                   const uint64_t *strides, const uint32_t *box)
{
    auto enc_t = encode_tiled_fn();
    if (!enc_t || rank < 2 || rank > 4) return false;
    cuuint64_t d[4], s[3];
    cuuint32_t b[4], estr[4] = {1, 1, 1, 1};
    TmapKey k;
    std::memset(&k, 0, sizeof k);
    k.kind = 2 + static_cast<uint32_t>(rank);
    k.type = static_cast<uint32_t>(type);
    k.ptr = reinterpret_cast<uint64_t>(ptr);
    for (int i = 0; i < rank; ++i) {
        d[i] = dims[i];
        b[i] = box[i];
        k.dims[i] = dims[i];
        k.box[i] = box[i];
        if (i + 1 < rank) {
            s[i] = strides[i];
            k.strides[i] = strides[i];
        }
    }
    return tmap_cached(k, m, [&](CUtensorMap *mm) {
        return enc_t(mm, type, static_cast<cuuint32_t>(rank), const_cast<void *>(ptr), d, s, b, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    });
}

// A 1x1, stride-1, unpadded layer reads x as a [B*H*W][C] matrix; any other
// layer reads x[B][H][W][C] through an im2col view.
int tc_x_tiled(const ConvArgs &a)
{
    return (a.KH == 1 && a.KW == 1 && a.sh == 1 && a.sw == 1 && a.ph == 0 && a.pw == 0) ? 1 : 0;
}

// Tensor map of the A operand: boxes of 128 output pixels x bk channels
// (128 bytes) in the 128-byte-swizzled K-major layout; im2col loads walk the
// output pixels across rows and images and read zeros in the padding.
bool tc_x_tmap(const ConvArgs &a, CUtensorMapDataType type, int elem, int bk, CUtensorMap *tmap_x)
{
    if (tc_x_tiled(a)) return tmap_2d(tmap_x, type, elem, a.x, static_cast<uint64_t>(a.B) * a.H * a.W, a.C, kBM);
    auto enc_i = encode_im2col_fn();
    if (!enc_i) return false;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(a.C), static_cast<cuuint64_t>(a.W),
                                static_cast<cuuint64_t>(a.H), static_cast<cuuint64_t>(a.B)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(a.C) * elem,
                                   static_cast<cuuint64_t>(a.C) * elem * a.W,
                                   static_cast<cuuint64_t>(a.C) * elem * a.W * a.H};
    int lower[2], upper[2];
    im2col_corners(a, lower, upper);
    const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(a.sw), static_cast<cuuint32_t>(a.sh), 1};
    TmapKey k;
    std::memset(&k, 0, sizeof k);
    k.kind = 1;
    k.type = static_cast<uint32_t>(type);
    k.ptr = reinterpret_cast<uint64_t>(a.x);
    for (int i = 0; i < 4; ++i) k.dims[i] = dims[i];
    for (int i = 0; i < 3; ++i) k.strides[i] = strides[i];
    for (int i = 0; i < 2; ++i) { k.lower[i] = lower[i]; k.upper[i] = upper[i]; }
    k.box[0] = static_cast<uint32_t>(bk); k.box[1] = kBM;
    for (int i = 0; i < 4; ++i) k.estr[i] = estr[i];
    return tmap_cached(k, tmap_x, [&](CUtensorMap *mm) {
        return enc_i(mm, type, 4, const_cast<void *>(a.x), dims, strides, lower, upper, bk, kBM, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    });
}

namespace {

template <typename Tr, int BN>
cudaError_t launch_bn(const ConvArgs &a, const typename Tr::T *W, const typename Tr::T *W_lo, void *sk_space,
                      cudaStream_t st, int split_s = 0, float *split_partials = nullptr)
{
    using L = TcLayout<Tr, BN>;
    constexpr int elem = sizeof(typename Tr::T);
    auto kern = tc_conv_kernel<Tr, BN>;
    const int K = a.KH * a.KW * a.C;
    auto enc_i = encode_im2col_fn();
    if (!enc_i) return cudaErrorNotSupported;
    // A: the activations' tensor map (none for the fused depthwise form,
    // whose A the split warps compute)
    const int a_tiled = tc_x_tiled(a);
    CUtensorMap tmap_x;
    if (a.dw_x) {
        std::memset(&tmap_x, 0, sizeof tmap_x);
    } else if (!tc_x_tmap(a, Tr::kTmap, elem, Tr::kBK, &tmap_x)) {
        return cudaErrorInvalidValue;
    }
    // B: W[C_out][K] (and W_lo), box 128 bytes of K x BN rows.  y:
    // [P_pix][C_out], stored in boxes of 128 bytes of columns x 32 rows, one
    // per epilogue warp (rows / columns outside y are not written).
    CUtensorMap tmap_w, tmap_wlo, tmap_y;
    if (!tmap_2d(&tmap_w, Tr::kTmap, elem, W, a.C_out, K, BN)) return cudaErrorInvalidValue;
    if (Tr::kSplit) {
        if (!tmap_2d(&tmap_wlo, Tr::kTmap, elem, W_lo, a.C_out, K, BN)) return cudaErrorInvalidValue;
    } else {
        tmap_wlo = tmap_w;                                     // unused
    }
    if (split_s > 0)
        tmap_y = tmap_w;                                       // split mode stores no y
    else if (!tmap_2d(&tmap_y, Tr::kTmap, elem, a.y, a.P_pix, a.C_out, 32))
        return cudaErrorInvalidValue;
    // the shared-memory opt-in, once per device for this kernel
    static std::mutex attr_mu;
    static bool attr_done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lk(attr_mu);
        if (!attr_done[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc);
            if (e != cudaSuccess) return e;
            attr_done[dev] = true;
        }
    }
    int sms = 0;
    e = device_sm_count(&sms);
    if (e != cudaSuccess) return e;
    TcSched sc{};
    sc.n_tn = (a.C_out + BN - 1) / BN;
    constexpr int kTileM = kBM * Tr::kMT;
    sc.n_tiles = ((a.P_pix + kTileM - 1) / kTileM) * sc.n_tn;
    const int n_cchunk = (a.C + Tr::kBK - 1) / Tr::kBK;
    sc.n_chunks = a.KH * a.KW * n_cchunk;
    sc.div_tn = FastDiv(static_cast<uint32_t>(sc.n_tn));
    sc.div_hw = FastDiv(static_cast<uint32_t>(a.Ho * a.Wo));
    sc.div_wo = FastDiv(static_cast<uint32_t>(a.Wo));
    sc.div_cchunk = FastDiv(static_cast<uint32_t>(n_cchunk));
    sc.div_kw = FastDiv(static_cast<uint32_t>(a.KW));
    int grid = sc.n_tiles < sms ? sc.n_tiles : sms;
    sc.dp_tiles = sc.n_tiles;
    // Stream-K for the last, partial round of tiles (all of them when there
    // are fewer tiles than SMs), with room for the partial slots: whole
    // rounds first, then the remaining tiles' chunk iterations spread over
    // the CTAs.  Each CTA gets at least kMinSplitIters chunk iterations and
    // at least C / kMaxParts of them, so that a split tile has at most
    // kMaxParts parts besides the finisher's.
    const int G = sms < kPlanCTAs ? sms : kPlanCTAs;
    if (split_s > 0) {
        if (split_s > sc.n_chunks || !split_partials) return cudaErrorInvalidValue;   // every item non-empty
        sc.split_s = split_s;
        sc.partials = split_partials;
        const int items = sc.n_tiles * split_s;
        grid = items < sms ? items : sms;
    } else if (sk_space && sc.n_tiles % G && sc.n_chunks >= sk_min_chunks(Tr::kSplit, Tr::kMT)) {
        const int dp = (sc.n_tiles / G) * G, skt = sc.n_tiles - dp;
        const int64_t iters = static_cast<int64_t>(skt) * sc.n_chunks;
        int need = (sc.n_chunks + L::kMaxParts - 1) / L::kMaxParts;
        if (need < kMinSplitIters) need = kMinSplitIters;
        const int gs = static_cast<int>(iters / need < G ? iters / need : G);
        if (gs > skt) {
            grid = dp ? G : gs;
            sc.dp_tiles = dp;
            sc.sk_tiles = skt;
            sc.sk_ctas = gs;
            sc.partials = static_cast<float *>(sk_space);
            sc.flags = reinterpret_cast<int *>(static_cast<unsigned char *>(sk_space) + sk_partial_bytes(BN, Tr::kMT));
        }
    }
    // Resident B: when the K loop fits in the stage ring, the column tile
    // of every tile of a CTA is the same (one column tile, or a grid that is
    // a multiple of their number, tiles dealt round-robin) and no tile is
    // split, each CTA loads its column tile's B chunks once, chunk c into
    // stage c's B region, and the stages then carry A only (ResNet-50's
    // 1x1 expansions re-read 2-4 B chunks of 32 KB per 128-row tile else).
    sc.b_resident = (sc.n_chunks <= L::kS && (sc.n_tn == 1 || grid % sc.n_tn == 0) && sc.sk_tiles == 0 &&
                     sc.split_s == 0)
                        ? 1
                        : 0;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(Tr::kWarps * 32);
    cfg.dynamicSmemBytes = L::kAlloc;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    // always a programmatic dependent of the previous kernel on the stream
    // (the decode, or the previous layer): the kernel touches global memory
    // only after griddepcontrol.wait
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a, tmap_x, tmap_w, tmap_wlo, tmap_y, sc, a_tiled);
}

// Column-tile width: the BN in {64, 128, 256} with the least estimated time,
// rounds of (SM count) tiles x a per-tile cost linear in BN (the MMA's N)
// plus a BN-independent share (A loads, epilogue start), 64 columns' worth.
// Narrow tiles win when there are few pixel tiles (more CTAs busy); wide
// tiles re-read the A operand fewer times.  Ties go to the wider tile.
// fp32 takes 128 instead of 256 unless that leaves a last column tile less
// than half full: at 256 the fp32 TMEM holds one accumulator next to the A
// ring, so a tile's MMAs wait for the previous tile's epilogue (measured on
// GB300: 3x3 512->512 on 128x14x14 472 -> 402 us, 1x1 96->576 33 -> 25 us;
// but 1x1 24->144, whose second 128-column tile would hold 16 columns,
// 83 -> 103 us).
int tc_bn(const ConvArgs &a, int dtype)
{
    const int64_t n_m = (static_cast<int64_t>(a.P_pix) + kBM - 1) / kBM;
    const int sms = device_sms_or_default();
    int best = 256;
    int64_t best_cost = -1;
    for (int bn : {256, 128, 64}) {
        if (bn > 64 && a.C_out <= bn / 2) continue;      // half the tile or more would be empty
        const int64_t tiles = n_m * ((a.C_out + bn - 1) / bn);
        const int64_t cost = ((tiles + sms - 1) / sms) * (bn + 64);
        if (best_cost < 0 || cost < best_cost) {
            best = bn;
            best_cost = cost;
        }
    }
    if (dtype == ONEXN_F32 && best == 256 && (a.C_out % 128 == 0 || a.C_out % 128 >= 64)) best = 128;
    return best;
}

// The im2col GEMM's tile.  Where the L2 -> SM stream of A and B tiles binds
// (bf16 layers with a long K loop: ~50-54 B per SM cycle on ResNet-50's
// stage-2 to -4 3x3 layers) and the 128-row plan takes 128 columns, tiles of
// 256 rows (two 128-row halves sharing each B tile) move a quarter fewer
// bytes per multiply-add (measured in the ResNet-50 stack: stage-4 3x3
// 55.5 -> 48.6 us, its stride-2 3x3 56.7 -> 49.3 us, stage-2 3x3 60.7 ->
// 58.2 us).  Taken for K loops of 32 or more chunks, and for stride-1
// spatial layers from 16 chunks; not for shorter K loops of 1x1 or strided
// layers (stage-2 1x1 512 -> 128 over 8 chunks 51.5 -> 65.3 us, stage-2
// stride-2 3x3 over 18 chunks 69.4 -> 79.3 us: the larger epilogue per tile
// and the stream-K fixup outweigh the bytes), nor at 256 columns: one
// 2 x 256-column accumulator fills the tensor memory, so every tile's (and
// stream-K piece's) epilogue stalls the next tile's MMAs (stage-3 3x3 46.8
// -> 62.5 us).
struct TcPlanTile {
    int bn, mt;
};
constexpr int kWideMinChunks = 16, kWideFewTilesMinChunks = 32;
TcPlanTile tc_plan_tile(const ConvArgs &a, int dtype)
{
    const int bn = tc_bn(a, dtype);
    const int n_chunks = a.KH * a.KW * ((a.C + TcBf16::kBK - 1) / TcBf16::kBK);
    const bool spatial_s1 = a.KH * a.KW > 1 && a.sh == 1 && a.sw == 1;
    const int64_t wide_tiles = ((static_cast<int64_t>(a.P_pix) + 2 * kBM - 1) / (2 * kBM)) * ((a.C_out + 127) / 128);
    const bool enough = wide_tiles >= 2 * static_cast<int64_t>(device_sms_or_default()) ||
                        n_chunks >= kWideFewTilesMinChunks;
    const bool wide = (spatial_s1 && n_chunks >= kWideMinChunks && enough) || n_chunks >= kWideFewTilesMinChunks;
    if (dtype == ONEXN_BF16 && bn == 128 && wide) return {128, 2};
    return {bn, 1};
}

size_t round256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

// decoded weights: bf16 C_out * K values; fp32 C_out * K values twice (hi, lo)
size_t weights_bytes(const ConvArgs &a, int dtype)
{
    const size_t n = static_cast<size_t>(a.C_out) * a.KH * a.KW * a.C;
    return round256(dtype == ONEXN_F32 ? n * 8 : n * 2);
}

// stream-K space after the weights: the partial slots, then the flags
size_t sk_bytes(const ConvArgs &a, int dtype)
{
    const TcPlanTile pt = tc_plan_tile(a, dtype);
    return sk_partial_bytes(pt.bn, pt.mt) + round256(kPlanCTAs * sizeof(int));
}

template <typename Tr>
cudaError_t decode_typed(const ConvArgs &a, void *workspace, size_t ws_bytes, cudaStream_t st)
{
    using T = typename Tr::T;
    const int K = a.KH * a.KW * a.C;
    const size_t n = static_cast<size_t>(a.C_out) * K;
    T *W = static_cast<T *>(workspace);
    T *W_lo = Tr::kSplit ? W + n : nullptr;
    const size_t wb = weights_bytes(a, Tr::kSplit ? ONEXN_F32 : ONEXN_BF16);
    int *flags = nullptr;
    const int dtype = Tr::kSplit ? ONEXN_F32 : ONEXN_BF16;
    if (ws_bytes >= wb + sk_bytes(a, dtype)) {
        const TcPlanTile pt = tc_plan_tile(a, dtype);
        flags = reinterpret_cast<int *>(static_cast<unsigned char *>(workspace) + wb +
                                        sk_partial_bytes(pt.bn, pt.mt));
    }
    const dim3 grid(static_cast<unsigned>((K + kDecodeCols - 1) / kDecodeCols), a.C_out / a.N,
                    (a.N + kDecodeRows - 1) / kDecodeRows);
    bsr_decode_kernel<T><<<grid, kDecodeCols, 0, st>>>(a.P, a.I, static_cast<const T *>(a.D), a.N, a.t, K, W, W_lo,
                                                        flags, kPlanCTAs);
    return cudaGetLastError();
}

template <typename Tr>
cudaError_t gemm_typed(const ConvArgs &a, const void *workspace, size_t ws_bytes, cudaStream_t st)
{
    using T = typename Tr::T;
    const size_t n = static_cast<size_t>(a.C_out) * a.KH * a.KW * a.C;
    const T *W = static_cast<const T *>(workspace);
    const T *W_lo = Tr::kSplit ? W + n : nullptr;
    const size_t wb = weights_bytes(a, Tr::kSplit ? ONEXN_F32 : ONEXN_BF16);
    const int dtype = Tr::kSplit ? ONEXN_F32 : ONEXN_BF16;
    void *sk = ws_bytes >= wb + sk_bytes(a, dtype)
                   ? static_cast<void *>(static_cast<unsigned char *>(const_cast<void *>(workspace)) + wb)
                   : nullptr;
    const TcPlanTile pt = tc_plan_tile(a, dtype);
    const int bn = pt.bn;
    // stride-1 spatial bf16 layers whose output rows fill the M tile: the
    // halo form loads each activation once per tile instead of once per tap
    if constexpr (!Tr::kSplit) {
        if (halo_form(a, bn) != kGemmIm2col) return halo_gemm(a, W, bn, st);
        if (pt.mt == 2) return launch_bn<TcBf16W, 128>(a, W, W_lo, sk, st);
    }
    if (bn == 64) return launch_bn<Tr, 64>(a, W, W_lo, sk, st);
    if (bn == 128) return launch_bn<Tr, 128>(a, W, W_lo, sk, st);
    return launch_bn<Tr, 256>(a, W, W_lo, sk, st);
}

}  // namespace

// Estimated time of the family (ns), for AUTO: the dense GEMM on the
// decoded weights (padded to whole tiles) at the machine rate measured on
// full-GPU layers (per multiply-add: fp32 as three tf32 products 7.9e-6 ns,
// bf16 2.3e-6 ns), scaled by SMs / the CTAs busy on average (fewer tiles,
// or stream-K pieces, than SMs; a ragged last round), plus fixed costs
// measured on GB300 against batch-1 layers: the GEMM's prologue, the
// stream-K fixup (partial tiles out, the finisher's wait and reads), and
// the decode launch unless the weights are already decoded.
double tc_cost_ns(const ConvArgs &a, int dtype, size_t ws_bytes, bool decoded)
{
    constexpr double kGemmFixedNs = 1200.0, kSkFixupNs = 7000.0, kDecodeFixedNs = 2000.0,
                     kDecodeBytesPerNs = 2000.0;
    const bool f32 = dtype == ONEXN_F32;
    const int bn = tc_bn(a, dtype);
    const int bk = f32 ? TcF32::kBK : TcBf16::kBK;
    const int64_t n_m = (static_cast<int64_t>(a.P_pix) + kBM - 1) / kBM, n_n = (a.C_out + bn - 1) / bn;
    const int64_t tiles = n_m * n_n, chunks = static_cast<int64_t>(a.KH) * a.KW * ((a.C + bk - 1) / bk);
    const size_t wb = weights_bytes(a, dtype);
    const int sms = device_sms_or_default();
    const int ctas = sms < kPlanCTAs ? sms : kPlanCTAs;
    const bool sk = ws_bytes >= wb + sk_bytes(a, dtype) && tiles < ctas && chunks >= sk_min_chunks(f32);
    double busy;
    if (tiles >= sms)
        busy = static_cast<double>(tiles) / static_cast<double>((tiles + sms - 1) / sms);
    else if (sk)
        busy = std::min<double>(ctas, static_cast<double>(tiles * chunks) / kMinSplitIters);
    else
        busy = static_cast<double>(tiles);
    const double dense = static_cast<double>(n_m * kBM) * static_cast<double>(n_n * bn) *
                         static_cast<double>(a.KH * a.KW * a.C);
    double ns = dense * (f32 ? 7.9e-6 : 2.3e-6) * sms / busy + kGemmFixedNs;
    if (sk) ns += kSkFixupNs;
    if (!decoded) ns += kDecodeFixedNs + static_cast<double>(wb) / kDecodeBytesPerNs;
    return ns;
}

// The decoded weights; with room for the stream-K partial slots and
// flags after them the GEMM also balances its last round of tiles.
size_t tc_workspace_min(const ConvArgs &a, int dtype) { return weights_bytes(a, dtype); }
size_t tc_workspace_bytes(const ConvArgs &a, int dtype) { return weights_bytes(a, dtype) + sk_bytes(a, dtype); }

// C_in, C_out giving 16-byte rows; the im2col box corners within the TMA's
// [-128, 127] range; strides <= 8; 16-bit tap offsets.
int tc_gemm_form(const ConvArgs &a, int dtype)
{
    const TcPlanTile pt = tc_plan_tile(a, dtype);
    if (dtype == ONEXN_BF16) {
        const int h = halo_form(a, pt.bn);
        if (h != kGemmIm2col) return h;
    }
    return pt.mt == 2 ? kGemmIm2colWide : kGemmIm2col;
}

bool tc_supports(const ConvArgs &a, int dtype)
{
    const int v = dtype == ONEXN_F32 ? 4 : 8;
    if (a.C % v || a.C_out % 8) return false;
    if (a.sh > 8 || a.sw > 8) return false;
    if (a.C_out / a.N > 65535) return false;          // decode grid.y
    int lower[2], upper[2];
    im2col_corners(a, lower, upper);
    for (int i = 0; i < 2; ++i)
        if (lower[i] < -128 || lower[i] > 127 || upper[i] < -128 || upper[i] > 127) return false;
    if ((a.KH - 1) * a.dh > 65535 || (a.KW - 1) * a.dw > 65535) return false;
    return true;
}

cudaError_t tc_decode(const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes, cudaStream_t st)
{
    return dtype == ONEXN_F32 ? decode_typed<TcF32>(a, workspace, ws_bytes, st)
                              : decode_typed<TcBf16>(a, workspace, ws_bytes, st);
}

namespace {
cudaError_t gemm_any(const ConvArgs &a, int dtype, const void *workspace, size_t ws_bytes, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    return dtype == ONEXN_F32 ? gemm_typed<TcF32>(a, workspace, ws_bytes, st)
                              : gemm_typed<TcBf16>(a, workspace, ws_bytes, st);
}
}  // namespace

cudaError_t tc_gemm(const ConvArgs &a, int dtype, const void *workspace, size_t ws_bytes, cudaStream_t st)
{
    return gemm_any(a, dtype, workspace, ws_bytes, st);
}

// ---- the GEMM on caller-given operands (the backward passes) ----

// The conv GEMM of `a` with the weights W (and W_lo for fp32) at explicit
// addresses instead of the workspace's decode: the input gradient runs the
// forward kernel on the flipped, transposed weights.
cudaError_t tc_gemm_weights(const ConvArgs &a, int dtype, const void *W, const void *W_lo, void *sk_space,
                            cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    const int bn = tc_bn(a, dtype);
    if (dtype == ONEXN_F32) {
        const float *w = static_cast<const float *>(W), *wl = static_cast<const float *>(W_lo);
        if (bn == 64) return launch_bn<TcF32, 64>(a, w, wl, sk_space, st);
        if (bn == 128) return launch_bn<TcF32, 128>(a, w, wl, sk_space, st);
        return launch_bn<TcF32, 256>(a, w, wl, sk_space, st);
    }
    const __nv_bfloat16 *w = static_cast<const __nv_bfloat16 *>(W);
    if (bn == 64) return launch_bn<TcBf16, 64>(a, w, w, sk_space, st);
    if (bn == 128) return launch_bn<TcBf16, 128>(a, w, w, sk_space, st);
    return launch_bn<TcBf16, 256>(a, w, w, sk_space, st);
}

// Plan of a split-mode GEMM C[M][N] = A[M][K] B[N][K]^T (K-major operands,
// K a multiple of 64): column tile BN, slices S (about one item per SM,
// at most one per K chunk) and the partial bytes (items x 128 x BN fp32).
TcSplitPlan tc_split_plan(int M, int Ncols, int64_t K, int dtype)
{
    TcSplitPlan p{};
    // the columns in as few tiles as possible: the slices, not narrow tiles,
    // spread the work over the SMs, and each column tile re-reads A
    p.bn = Ncols <= 64 ? 64 : Ncols <= 128 ? 128 : 256;
    const int64_t tiles = ((static_cast<int64_t>(M) + kBM - 1) / kBM) * ((Ncols + p.bn - 1) / p.bn);
    const int64_t chunks = (K + (dtype == ONEXN_F32 ? TcF32::kBK : TcBf16::kBK) - 1) /
                           (dtype == ONEXN_F32 ? TcF32::kBK : TcBf16::kBK);
    int64_t S = device_sms_or_default() / (tiles > 0 ? tiles : 1);
    if (S < 1) S = 1;
    if (S > chunks) S = chunks > 0 ? chunks : 1;
    p.tiles = static_cast<int>(tiles);
    p.n_tn = (Ncols + p.bn - 1) / p.bn;
    p.split_s = static_cast<int>(S);
    p.partial_bytes = static_cast<size_t>(tiles * S) * kBM * p.bn * 4;
    return p;
}

// The split-mode GEMM: A = x [M][K] (a.x), B = W [N][K] (and W_lo), the
// item accumulators into partials (plan.partial_bytes).
cudaError_t tc_gemm_split(const ConvArgs &a, int dtype, const void *W, const void *W_lo, float *partials,
                          const TcSplitPlan &plan, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    if (dtype == ONEXN_F32) {
        const float *w = static_cast<const float *>(W), *wl = static_cast<const float *>(W_lo);
        if (plan.bn == 64) return launch_bn<TcF32, 64>(a, w, wl, nullptr, st, plan.split_s, partials);
        if (plan.bn == 128) return launch_bn<TcF32, 128>(a, w, wl, nullptr, st, plan.split_s, partials);
        return launch_bn<TcF32, 256>(a, w, wl, nullptr, st, plan.split_s, partials);
    }
    const __nv_bfloat16 *w = static_cast<const __nv_bfloat16 *>(W);
    if (plan.bn == 64) return launch_bn<TcBf16, 64>(a, w, w, nullptr, st, plan.split_s, partials);
    if (plan.bn == 128) return launch_bn<TcBf16, 128>(a, w, w, nullptr, st, plan.split_s, partials);
    return launch_bn<TcBf16, 256>(a, w, w, nullptr, st, plan.split_s, partials);
}

size_t tc_weights_bytes(const ConvArgs &a, int dtype) { return weights_bytes(a, dtype); }
size_t tc_sk_bytes(const ConvArgs &a, int dtype) { return sk_bytes(a, dtype); }

// decode, then the GEMM as its programmatic dependent (its launch and
// prologue overlap the decode)
cudaError_t launch_tc(const ConvArgs &a, int dtype, void *workspace, size_t ws_bytes, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    const cudaError_t e = tc_decode(a, dtype, workspace, ws_bytes, st);
    return e != cudaSuccess ? e : gemm_any(a, dtype, workspace, ws_bytes, st);
}

}  // namespace onexn
