// Sparse tensor-core (tcgen05) kernel of the 1xN-pruned convolution, bf16:
// Eq. 7 computed block by block on the tensor cores, so that only the kept
// blocks are multiplied.
//
// Each output group g (N consecutive output channels) contracts over its
// own kept list I[P_g .. P_{g+1}) (Sec. 3.4).  Per tile of 128 output
// pixels and GS = 128 / N groups the K walk is the same as the dense
// kernel's: chunks of one filter tap x 64 input channels, loaded by TMA
// (im2col) into shared memory.  Each chunk is gathered in two halves of 32
// channels.  For a half, group g's kept entries z (a contiguous range of
// its list, since I is increasing) are copied column by column from the
// staged activations into a per-group A block in tensor memory (lane =
// output pixel, 32-bit column = two consecutive kept entries), padded with
// zeros to a multiple of 16 entries, and their weight rows D[z][0..N) are
// staged as the K-major B operand.  One tcgen05.mma of M = 128, N, K = 16
// then multiplies 16 kept entries of one group: the tensor work is the kept
// work rounded up to 16 entries per group and half-chunk, not the dense
// work of the decoded layer.
//
// Warp roles (one persistent CTA per SM):
//  * warp 2, producer: one thread issues the TMA load of each chunk's
//    activation tile (128 pixels x 64 channels, 128-byte swizzle) and one
//    bulk copy of the chunk's plan record, which a plan kernel wrote once
//    per layer with the kept entries' channels and their D rows, so no load
//    depends on another.
//  * warps 4-11, gather: warp w handles pixel rows 32*(w%4) .. +31 of the
//    tile (its TMEM lanes) and half-chunk (w-4)/4.  Per chunk and group it
//    reads the entries' input channels from I, copies x[row][c] into the
//    group's A block with tcgen05.st, and (warp g%4 of the half) writes the
//    group's D rows into B and its entry count into shared memory; then
//    arrives on "gathered" of its half.
//  * warps 0-1, MMA: lane 0 of warp q issues the MMAs of groups g = q mod 2
//    (two issuing threads, since one thread's back-to-back tcgen05.mma of
//    N = 16 issue about one per 45 cycles) and commits them; warp 0 owns
//    the TMEM allocation.
//  * warps 12-15, epilogue: read the tile's accumulators, add the bias (and
//    residual), apply the activation and store bf16 NHWC.
// Every wait is bounded (about one second); on expiry the kernel sets the
// status word, stops, drains its MMAs and frees the TMEM.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "onexn_internal.h"
#include "tc_maps.h"
#include "tc_ptx.cuh"

#include <mutex>

namespace onexn {

namespace {

constexpr int kBM = 128;                   // output pixels per tile (TMEM lanes, UMMA M)
constexpr int kTileCols = 128;             // output columns per tile: GS groups x N
constexpr int kMaxGS = 8;                  // groups per tile at most (N = 16)
constexpr int kBK = 64;                    // channels per chunk (128 bytes of bf16)
constexpr int kHalf = 32;                  // channels per gathered half-chunk
constexpr int kStages = 4;
// plan record of one (chunk, group tile), built once per layer:
//   [0, 16)   uint8 count[h * 8 + gl]   kept entries of group g0+gl in half-chunk h (<= 32)
//   [16, 48)  int32 zs[gl]              first entry of the chunk in the group's list
//   [48, 560) uint8 ch[(h*8 + gl)*32 + j]  channel of entry j inside half-chunk h (0..31)
//   [560, +kDBytes) the D rows of those entries: group gl's at gl * 64 * N
//             bf16, half 0's entries then half 1's, N values each
// so that one copy per chunk brings everything its gathers and MMAs read.
constexpr int kRecCnt = 0, kRecZs = 16, kRecCh = 48, kRecHdr = 560;
constexpr int kXBytes = kBM * 128;                   // 128 pixels x 64 channels, 128-byte swizzle
constexpr int kBBytes = kTileCols * 128;             // per group N rows x 64 entries, K-major, 128-byte swizzle
constexpr int kDBytes = kTileCols * kBK * 2;         // per group up to 64 rows of N bf16
constexpr int kRecBytes = kRecHdr + kDBytes;         // a multiple of 16 (bulk copy)
// stage: activation tile | B of the tile's groups | record (its D rows inside)
constexpr int kXOff = 0, kBOff = kXBytes, kRecOff = kBOff + kBBytes, kDOff = kRecOff + kRecHdr;
constexpr int kStageBytes = ((kRecOff + kRecBytes + 1023) / 1024) * 1024;
static_assert(kRecBytes % 16 == 0 && kDOff % 16 == 0, "bulk copy and 16-byte D row loads");
constexpr int kAccCols = kTileCols;        // one fp32 accumulator buffer; two of them
constexpr int kACol0 = 2 * kAccCols;       // A blocks after the accumulators: [half][group]
constexpr int kABlockCols = 16;            // per (half, group): 32 bf16 entries per lane
constexpr int kTmemCols = 512;
constexpr int kIssuers = 2;                // warps 0, 1
constexpr int kProdWarp = 2;               // warp 3 has no role
constexpr int kGather0 = 4;                // warps 4..7: half 0; warps 8..11: half 1
constexpr int kEpi0 = 12;                  // warps 12..15
constexpr int kWarps = 16;

// shared memory (from a 1024-byte aligned base)
constexpr int kXtWarpBytes = 16 * 32 * 4;  // a gather warp's transposed half rows: 16 words x 32 lanes
constexpr int kXtOff = kStages * kStageBytes;
constexpr int kBarOff = kXtOff + 8 * kXtWarpBytes;
// full[S], empty[S], gathered[2], consumed[2], tfull[2], tempty[2], drain[kIssuers]
constexpr int kNumBars = 2 * kStages + 2 + 2 + 2 + 2 + kIssuers;
constexpr int kMaskOff = kBarOff + kNumBars * 8;       // uint32 [2][kIssuers]: groups an issuer touched
constexpr int kHolderOff = kMaskOff + 2 * kIssuers * 4;
constexpr int kSmemBytes = kHolderOff + 16;
constexpr int kSmemAlloc = kSmemBytes + 1024;

static_assert(kACol0 + 2 * kMaxGS * kABlockCols <= kTmemCols, "tensor memory");
static_assert(kSmemAlloc <= 232448, "shared memory");

struct MmaSched {
    int n_g;             // group tiles (ceil(G / GS))
    int tiles;           // pixel tiles x group tiles
    int G;               // groups of the layer
    int n_cchunk;        // 64-channel chunks per tap
    int n_chunks;        // taps x n_cchunk
    FastDiv div_g, div_hw, div_wo, div_cchunk, div_kw;
    const unsigned char *rec;   // [n_chunks][n_g] records of kRecBytes
};

// first z in [lo, hi) with I[z] >= k (I increasing in that range)
__device__ __forceinline__ int lower_bound_k(const int32_t *__restrict__ I, int lo, int hi, int64_t k)
{
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(I + mid) < k) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// The plan records: for chunk ci (tap, 64-channel block), group tile tg and
// half-chunk h, the kept entries z of group g = tg*GS + gl whose index
// I[z] = tap*C + c has c in the half-chunk's 32 channels (a contiguous
// range of the group's list, found by binary search), their count and
// channels, their D rows (after the chunk's half-0 rows); and the chunk's
// first entry.  P and I are clamped so that a corrupted list cannot index
// outside I or D.  One thread per (ci, tg, gl, h).
__global__ void mma_plan_kernel(const int32_t *__restrict__ P, const int32_t *__restrict__ I,
                                const __nv_bfloat16 *__restrict__ D, int N, int t, int G, int GS, int C,
                                int n_cchunk, int n_chunks, int n_g, unsigned char *__restrict__ rec)
{
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<int64_t>(n_chunks) * n_g * GS * 2) return;
    const int h = static_cast<int>(idx & 1);
    const int64_t r1 = idx >> 1;
    const int gl = static_cast<int>(r1 % GS);
    const int64_t r2 = r1 / GS;
    const int tg = static_cast<int>(r2 % n_g), ci = static_cast<int>(r2 / n_g);
    unsigned char *r = rec + (static_cast<int64_t>(ci) * n_g + tg) * kRecBytes;
    const int g = tg * GS + gl;
    int z0 = 0, cnt = 0;
    const int tap = ci / n_cchunk, cc = ci - tap * n_cchunk;
    const int c_lo = min(C, cc * kBK + h * kHalf), c_hi = min(C, cc * kBK + (h + 1) * kHalf);
    const int64_t kbase = static_cast<int64_t>(tap) * C + cc * kBK + h * kHalf;
    if (g < G) {
        const int lo = clampi(__ldg(P + g), 0, t), hi = clampi(__ldg(P + g + 1), lo, t);
        z0 = lower_bound_k(I, lo, hi, static_cast<int64_t>(tap) * C + c_lo);
        const int z1 = lower_bound_k(I, z0, hi, static_cast<int64_t>(tap) * C + c_hi);
        cnt = min(z1 - z0, kHalf);
        if (h == 0) reinterpret_cast<int32_t *>(r + kRecZs)[gl] = z0;
        // D rows of this half's entries: after the chunk's half-0 entries
        const int zc = h ? lower_bound_k(I, lo, z0, static_cast<int64_t>(tap) * C + cc * kBK) : z0;
        const int off = min(z0 - zc, kHalf);
        const uint4 *src = reinterpret_cast<const uint4 *>(D + static_cast<int64_t>(z0) * N);
        uint4 *dst = reinterpret_cast<uint4 *>(r + kRecHdr + gl * (kBK * N * 2) + off * (N * 2));
        for (int i = 0; i < cnt * (N / 8); ++i) dst[i] = __ldg(src + i);
    } else if (h == 0) {
        reinterpret_cast<int32_t *>(r + kRecZs)[gl] = 0;
    }
    r[kRecCnt + h * kMaxGS + gl] = static_cast<unsigned char>(cnt);
    unsigned char *ch = r + kRecCh + (h * kMaxGS + gl) * kHalf;
    for (int j = 0; j < kHalf; ++j)
        ch[j] = static_cast<unsigned char>(j < cnt ? clampi(static_cast<int>(__ldg(I + z0 + j) - kbase), 0, kHalf - 1) : 0);
}

__device__ __forceinline__ void sts_u16(uint32_t addr, uint32_t v)
{
    asm volatile("st.shared.u16 [%0], %1;\n" ::"r"(addr), "h"(static_cast<unsigned short>(v)) : "memory");
}

// byte offset of (row, entry) in a K-major tile of 64-entry (128-byte) rows
// with the 128-byte swizzle: 16-byte chunk j of row r sits at chunk j ^ (r % 8)
__device__ __forceinline__ uint32_t sw128(int row, int e)
{
    return static_cast<uint32_t>(row * 128 + ((((e >> 3) ^ (row & 7))) << 4) + ((e & 7) << 1));
}

template <int N>
__global__ void __launch_bounds__(kWarps * 32, 1)
mma_conv_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_x, const MmaSched sc, const int a_tiled)
{
    constexpr int GS = kTileCols / N;              // groups per tile
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    const uint32_t bar_full = base + kBarOff;
    const uint32_t bar_empty = bar_full + 8 * kStages;
    const uint32_t bar_gath = bar_empty + 8 * kStages;
    const uint32_t bar_cons = bar_gath + 16;
    const uint32_t bar_tfull = bar_cons + 16;
    const uint32_t bar_tempty = bar_tfull + 16;
    const uint32_t bar_drain = bar_tempty + 16;
    uint32_t *mask_tab = reinterpret_cast<uint32_t *>(smem + kMaskOff);
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + kHolderOff);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(bar_full + 8 * s, 1);
            mbar_init(bar_empty + 8 * s, kIssuers);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar_gath + 8 * b, 128);
            mbar_init(bar_cons + 8 * b, kIssuers);
            mbar_init(bar_tfull + 8 * b, 2 * kIssuers);   // each issuer: its MMAs' commit + its mask
            mbar_init(bar_tempty + 8 * b, 128);
        }
        for (int q = 0; q < kIssuers; ++q) mbar_init(bar_drain + 8 * q, 1);
        fence_mbar_init();
    }
    // B entries that no kept block fills are multiplied by zero A entries;
    // they start as zeros (finite) and later hold earlier weights
    for (int s = 0; s < kStages; ++s)
        for (int i = tid; i < kBBytes / 16; i += kWarps * 32)
            reinterpret_cast<uint4 *>(smem + s * kStageBytes + kBOff)[i] = make_uint4(0u, 0u, 0u, 0u);
    tc::fence_proxy_async_smem();
    if (warp == 0) {
        tc::tmem_alloc(smem_u32(holder), kTmemCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;
    auto abort_now = [&]() { atomicOr(a.status, kStatusTimeout); };
    const int G = sc.G;

    if (warp == kProdWarp) {
        // ============================ producer ============================
        // Per chunk: the activation tile (TMA) and the chunk's plan record,
        // its D rows inside (one bulk copy), both on "full".
        if (lane == 0) {
            const int hw = a.Ho * a.Wo;
            bool failed = false;
            int item = 0;
            for (int T = blockIdx.x; T < sc.tiles && !failed; T += gridDim.x) {
                const int tm = static_cast<int>(sc.div_g.div(T)), tg = T - tm * sc.n_g;
                const int p0 = tm * kBM;
                const int b0 = static_cast<int>(sc.div_hw.div(p0)), r0 = p0 - b0 * hw;
                const int oh0 = static_cast<int>(sc.div_wo.div(r0)), ow0 = r0 - oh0 * a.Wo;
                const int w0 = ow0 * a.sw - a.pw, h0 = oh0 * a.sh - a.ph;
                for (int ci = 0; ci < sc.n_chunks; ++ci, ++item) {
                    const int s = item % kStages;
                    if (item >= kStages && !mbar_wait(bar_empty + 8 * s, ((item / kStages) + 1) & 1)) {
                        failed = true;
                        break;
                    }
                    const int tap = static_cast<int>(sc.div_cchunk.div(ci)), cc = ci - tap * sc.n_cchunk;
                    const int kh = static_cast<int>(sc.div_kw.div(tap)), kw = tap - kh * a.KW;
                    const uint32_t xs = base + s * kStageBytes + kXOff;
                    tc::mbar_arrive_expect_tx(bar_full + 8 * s, kXBytes + kRecBytes);
                    if (a_tiled)
                        tc::tma_load_2d(xs, &tmap_x, cc * kBK, p0, bar_full + 8 * s);
                    else
                        tc::tma_load_im2col_4d(xs, &tmap_x, cc * kBK, w0, h0, b0, static_cast<uint16_t>(kw * a.dw),
                                               static_cast<uint16_t>(kh * a.dh), bar_full + 8 * s);
                    tc::bulk_load(base + s * kStageBytes + kRecOff,
                                  sc.rec + (static_cast<int64_t>(ci) * sc.n_g + tg) * kRecBytes, kRecBytes,
                                  bar_full + 8 * s);
                }
            }
            if (failed) abort_now();
        }
        __syncwarp();
    } else if (warp >= kGather0 && warp < kGather0 + 8) {
        // ============================= gather =============================
        // Warp (q, h) = (w % 4, (w - 4) / 4): thread i owns pixel row 32q + i
        // of the tile (TMEM lane) and half-chunk h (channels 32h .. 32h+31 of
        // every chunk).  Per chunk it copies its row's half into its column of
        // a warp-private transposed buffer (word u of lane l at u*32 + l),
        // from which the per-entry reads hit 32 distinct banks; then, group by
        // group, it reads the kept entries' channels from the plan record,
        // packs pairs of x[row][c] into 32-bit words and stores them to the
        // group's A block with tcgen05.st.  Warp g % 4 of the half then writes
        // group g's D rows into its B block.
        const int q = warp & 3, h = (warp - kGather0) >> 2;
        const int row = 32 * q + lane;
        const uint32_t lane_t = tmem + (static_cast<uint32_t>(32 * q) << 16);
        uint32_t *xt = reinterpret_cast<uint32_t *>(smem + kXtOff + (warp - kGather0) * kXtWarpBytes) + lane;
        constexpr int V = N / 8;                          // 16-byte vectors per D row
        int item = 0;
        bool failed = false;
        for (int T = blockIdx.x; T < sc.tiles && !failed; T += gridDim.x) {
            const int tm = static_cast<int>(sc.div_g.div(T)), tg = T - tm * sc.n_g;
            const int g0 = tg * GS;
            for (int ci = 0; ci < sc.n_chunks; ++ci, ++item) {
                const int s = item % kStages;
                if (!mbar_wait(bar_full + 8 * s, (item / kStages) & 1)) {
                    abort_now();
                    failed = true;
                    break;
                }
                const uint32_t st0 = base + s * kStageBytes;
                const unsigned char *r = smem + s * kStageBytes + kRecOff;
                // this thread's half row -> its column of the transposed buffer
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    uint32_t v0, v1, v2, v3;
                    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];\n"
                                 : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
                                 : "r"(st0 + kXOff + row * 128 + (((4 * h + j) ^ (row & 7)) << 4))
                                 : "memory");
                    xt[(4 * j) * 32] = v0;
                    xt[(4 * j + 1) * 32] = v1;
                    xt[(4 * j + 2) * 32] = v2;
                    xt[(4 * j + 3) * 32] = v3;
                }
                // the A blocks of this half are free once the MMAs of the
                // previous chunk's half h have completed
                if (item >= 1 && !mbar_wait(bar_cons + 8 * h, (item - 1) & 1)) {
                    abort_now();
                    failed = true;
                    break;
                }
                tc::fence_after_sync();
#pragma unroll
                for (int g = 0; g < GS; ++g) {
                    const int cnt = (g0 + g < G) ? r[kRecCnt + h * kMaxGS + g] : 0;
                    const int cw = r[kRecCh + (h * kMaxGS + g) * kHalf + lane] & (kHalf - 1);
                    const int pk = ((cw >> 1) << 6) | (cw & 1);     // (word * 32 lanes) << 1 | half
                    const int nb = (cnt + 15) >> 4;
                    for (int bb = 0; bb < nb; ++bb) {
                        int pj[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) pj[i] = __shfl_sync(0xffffffffu, pk, 16 * bb + i);
                        uint32_t vv[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) vv[i] = (16 * bb + i < cnt) ? xt[pj[i] >> 1] : 0u;
                        uint32_t w[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i)
                            w[i] = __byte_perm(vv[2 * i], vv[2 * i + 1],
                                               ((pj[2 * i] & 1) ? 0x32u : 0x10u) | ((pj[2 * i + 1] & 1) ? 0x7600u : 0x5400u));
                        tc::st_32x32b_x8(lane_t + kACol0 + (h * GS + g) * kABlockCols + 8 * bb, w);
                    }
                }
                // the staged groups' B: entry j of the half -> K position
                // 32h + j of rows n = 0..N-1 (from the group's D rows in this
                // stage's copy of the record, after the half-0 entries for
                // h = 1); the rest of each used 16-entry step is zeroed
                for (int g = q; g < GS; g += 4) {
                    if (g0 + g >= G) break;
                    const int cnt = r[kRecCnt + h * kMaxGS + g], nb = (cnt + 15) >> 4;
                    const int off = h ? r[kRecCnt + g] : 0;
                    const uint32_t bg = st0 + kBOff + g * N * 128;
                    const uint32_t dg = st0 + kDOff + g * (kBK * N * 2) + off * (N * 2);
                    for (int idx = lane; idx < 16 * nb * V; idx += 32) {
                        const int j = idx / V, v = idx - j * V;
                        uint32_t d0 = 0u, d1 = 0u, d2 = 0u, d3 = 0u;
                        if (j < cnt)
                            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];\n"
                                         : "=r"(d0), "=r"(d1), "=r"(d2), "=r"(d3)
                                         : "r"(dg + j * (N * 2) + v * 16)
                                         : "memory");
                        const uint32_t dv[4] = {d0, d1, d2, d3};
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            sts_u16(bg + sw128(8 * v + e, 32 * h + j), (dv[e >> 1] >> (16 * (e & 1))) & 0xffffu);
                    }
                }
                tc::st_wait();
                tc::fence_proxy_async_smem();
                tc::fence_before_sync();
                mbar_arrive(bar_gath + 8 * h);
            }
        }
    } else if (warp < kIssuers) {
        // =============================== MMA ===============================
        if (lane == 0) {
            const int q = warp;
            constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, N);
            int item = 0, ti = 0;
            bool failed = false;
            for (int T = blockIdx.x; T < sc.tiles && !failed; T += gridDim.x, ++ti) {
                const int tm = static_cast<int>(sc.div_g.div(T)), tg = T - tm * sc.n_g;
                const int g0 = tg * GS;
                const int acc = ti & 1, use = ti >> 1;
                if (use >= 1 && !mbar_wait(bar_tempty + 8 * acc, (use - 1) & 1)) {
                    abort_now();
                    break;
                }
                tc::fence_after_sync();
                uint32_t touched = 0;
                const uint32_t d_base = tmem + acc * kAccCols;
                for (int ci = 0; ci < sc.n_chunks && !failed; ++ci, ++item) {
                    const int s = item % kStages;
                    const uint32_t bs = base + s * kStageBytes + kBOff;
                    const unsigned char *r = smem + s * kStageBytes + kRecOff;
                    for (int h = 0; h < 2; ++h) {
                        if (!mbar_wait(bar_gath + 8 * h, item & 1)) {
                            abort_now();
                            failed = true;
                            break;
                        }
                        tc::fence_after_sync();
                        for (int g = q; g < GS && g0 + g < G; g += kIssuers) {
                            const int nb = (r[kRecCnt + h * kMaxGS + g] + 15) >> 4;
                            const uint64_t bd = tc::desc_kmajor_sw128(bs + g * N * 128);
                            for (int bb = 0; bb < nb; ++bb) {
                                tc::mma_bf16_ta(d_base + g * N, tmem + kACol0 + (h * GS + g) * kABlockCols + 8 * bb,
                                                bd + 2 * (2 * h + bb), idesc, (touched >> g) & 1u);
                                touched |= 1u << g;
                            }
                        }
                        tc::commit(bar_cons + 8 * h);
                    }
                    if (!failed) tc::commit(bar_empty + 8 * s);
                }
                if (failed) break;
                mask_tab[acc * kIssuers + q] = touched;
                tc::commit(bar_tfull + 8 * acc);
                mbar_arrive(bar_tfull + 8 * acc);
            }
            // everything this thread issued completes before the TMEM is freed
            tc::commit(bar_drain + 8 * q);
            if (!mbar_wait(bar_drain + 8 * q, 0)) abort_now();
        }
        __syncwarp();
    } else if (warp >= kEpi0 && warp < kEpi0 + 4) {
        // ============================ epilogue ============================
        const int q = warp & 3;
        const int row = 32 * q + lane;
        const uint32_t lane_t = tmem + (static_cast<uint32_t>(32 * q) << 16);
        __nv_bfloat16 *y = static_cast<__nv_bfloat16 *>(a.y);
        const __nv_bfloat16 *res = static_cast<const __nv_bfloat16 *>(a.residual);
        int ti = 0;
        for (int T = blockIdx.x; T < sc.tiles; T += gridDim.x, ++ti) {
            const int acc = ti & 1;
            if (!mbar_wait(bar_tfull + 8 * acc, (ti >> 1) & 1)) {
                abort_now();
                break;
            }
            tc::fence_after_sync();
            uint32_t touched = 0;
#pragma unroll
            for (int i = 0; i < kIssuers; ++i) touched |= mask_tab[acc * kIssuers + i];
            const int tm = static_cast<int>(sc.div_g.div(T)), tg = T - tm * sc.n_g;
            const int g0 = tg * GS;
            const int p = tm * kBM + row;
            for (int g = 0; g < GS && g0 + g < G; ++g) {
                const int col0 = (g0 + g) * N;
                const bool on = (touched >> g) & 1u;
                __nv_bfloat16 *yr = y + static_cast<int64_t>(p) * a.C_out + col0;
#pragma unroll 1
                for (int pc = 0; pc < N / 16; ++pc) {
                    uint32_t r[16];
                    tc::ld_32x32b_x16(lane_t + acc * kAccCols + g * N + 16 * pc, r);
                    tc::ld_wait();
                    if (p >= a.P_pix) continue;
#pragma unroll
                    for (int v = 0; v < 2; ++v) {
                        const int n0 = 16 * pc + 8 * v;
                        float o[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            o[e] = (on ? __uint_as_float(r[8 * v + e]) : 0.f) + (a.bias ? __ldg(a.bias + col0 + n0 + e) : 0.f);
                        if (res) {
                            const uint4 rv = __ldg(reinterpret_cast<const uint4 *>(
                                res + static_cast<int64_t>(p) * a.C_out + col0 + n0));
                            const uint32_t rw[4] = {rv.x, rv.y, rv.z, rv.w};
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                o[2 * e] += bf16lo(rw[e]);
                                o[2 * e + 1] += bf16hi(rw[e]);
                            }
                        }
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[e] = activate(o[e], a.relu);
                        reinterpret_cast<uint4 *>(yr + n0)[0] = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                                                                           pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
                    }
                }
            }
            tc::fence_before_sync();
            mbar_arrive(bar_tempty + 8 * acc);
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

int n_cchunk_of(const ConvArgs &a) { return (a.C + kBK - 1) / kBK; }
int n_chunks_of(const ConvArgs &a) { return a.KH * a.KW * n_cchunk_of(a); }
int gs_of(const ConvArgs &a) { return kTileCols / a.N; }
int n_g_of(const ConvArgs &a) { return (a.C_out / a.N + gs_of(a) - 1) / gs_of(a); }

template <int N>
cudaError_t launch_n(const ConvArgs &a, const unsigned char *rec, cudaStream_t st)
{
    auto kern = mma_conv_kernel<N>;
    CUtensorMap tmap_x;
    if (!tc_x_tmap(a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, kBK, &tmap_x)) return cudaErrorInvalidValue;
    static std::mutex attr_mu;
    static bool attr_done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lk(attr_mu);
        if (!attr_done[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemAlloc);
            if (e != cudaSuccess) return e;
            attr_done[dev] = true;
        }
    }
    int sms = 0;
    e = device_sm_count(&sms);
    if (e != cudaSuccess) return e;
    MmaSched sc{};
    sc.G = a.C_out / a.N;
    sc.n_g = n_g_of(a);
    sc.tiles = ((a.P_pix + kBM - 1) / kBM) * sc.n_g;
    sc.n_cchunk = n_cchunk_of(a);
    sc.n_chunks = n_chunks_of(a);
    sc.div_g = FastDiv(static_cast<uint32_t>(sc.n_g));
    sc.div_hw = FastDiv(static_cast<uint32_t>(a.Ho * a.Wo));
    sc.div_wo = FastDiv(static_cast<uint32_t>(a.Wo));
    sc.div_cchunk = FastDiv(static_cast<uint32_t>(sc.n_cchunk));
    sc.div_kw = FastDiv(static_cast<uint32_t>(a.KW));
    sc.rec = rec;
    const int grid = sc.tiles < sms ? sc.tiles : sms;
    kern<<<grid, kWarps * 32, kSmemAlloc, st>>>(a, tmap_x, sc, tc_x_tiled(a));
    return cudaGetLastError();
}

size_t round256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

}  // namespace

// The plan: one record of kRecBytes per (chunk, group tile).
size_t mma_workspace_bytes(const ConvArgs &a)
{
    return round256(static_cast<size_t>(n_chunks_of(a)) * n_g_of(a) * kRecBytes);
}

// bf16 (checked by the caller), N a multiple of 16 up to 128 (one MMA of
// M = 128, N per 16 kept entries of a group), and what the dense kernel's
// activation loads need (16-byte rows, TMA im2col bounds).
bool mma_supports(const ConvArgs &a)
{
    if (a.N != 16 && a.N != 32 && a.N != 64 && a.N != 128) return false;
    return tc_supports(a, ONEXN_BF16);
}

// Writes the plan into the workspace.
cudaError_t mma_plan(const ConvArgs &a, void *workspace, size_t ws_bytes, cudaStream_t st)
{
    if (!workspace || ws_bytes < mma_workspace_bytes(a)) return cudaErrorInvalidValue;
    const int G = a.C_out / a.N, GS = gs_of(a), n_g = n_g_of(a), n_chunks = n_chunks_of(a);
    const int64_t n = static_cast<int64_t>(n_chunks) * n_g * GS * 2;
    const int threads = 256;
    mma_plan_kernel<<<static_cast<unsigned>((n + threads - 1) / threads), threads, 0, st>>>(
        a.P, a.I, static_cast<const __nv_bfloat16 *>(a.D), a.N, a.t, G, GS, a.C, n_cchunk_of(a), n_chunks, n_g,
        static_cast<unsigned char *>(workspace));
    return cudaGetLastError();
}

// The kernel on a plan already in the workspace.
cudaError_t mma_run(const ConvArgs &a, const void *workspace, size_t ws_bytes, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    if (!workspace || ws_bytes < mma_workspace_bytes(a)) return cudaErrorInvalidValue;
    const unsigned char *rec = static_cast<const unsigned char *>(workspace);
    switch (a.N) {
    case 16: return launch_n<16>(a, rec, st);
    case 32: return launch_n<32>(a, rec, st);
    case 64: return launch_n<64>(a, rec, st);
    case 128: return launch_n<128>(a, rec, st);
    default: return cudaErrorNotSupported;
    }
}

cudaError_t launch_mma(const ConvArgs &a, void *workspace, size_t ws_bytes, cudaStream_t st)
{
    if (a.P_pix == 0) return cudaSuccess;
    const cudaError_t e = mma_plan(a, workspace, ws_bytes, st);
    return e != cudaSuccess ? e : mma_run(a, workspace, ws_bytes, st);
}

}  // namespace onexn
