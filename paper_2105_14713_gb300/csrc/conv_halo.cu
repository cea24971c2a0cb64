// Tensor-core GEMM of stride-1 spatial convolutions (bf16) on halo tiles.
//
// The im2col form of the tcgen05 GEMM (conv_tc.cu) loads a fresh A tile of
// 128 output pixels for every tap and the B tile of that tap for every
// pixel tile, so a 3x3 layer moves each activation nine times and its
// weights once per tile from L2 into shared memory.  Here:
//  * a tile is R whole output rows of one image, laid out along M with the
//    padded row width Wp = Wo + (KW-1)*dw: M row m is output pixel
//    (h0 + m / Wp, m % Wp); rows with m % Wp >= Wo or past the tile's rows
//    are computed and dropped;
//  * per 64-channel chunk one TMA im2col load brings the Wp x Rh input
//    positions of rows h0 - ph .. h0 - ph + R + (KH-1)*dh - 1, columns
//    -pw .. -pw + Wp - 1 (zeros outside the image), one 128-byte swizzled
//    row per position, and the A operand of tap (kh, kw) is that buffer
//    viewed from row kh*dh*Wp + kw*dw on: output pixel (r, w) of the tile
//    reads input position (r + kh*dh, w + kw*dw) of the halo.  The swizzle
//    is a function of the shared-memory address, so a view may start at any
//    128-byte row;
//  * each CTA serves one column tile of BN output channels, whose decoded
//    weights (all taps and chunks) it loads once and keeps in shared memory.
// The sum over taps and chunks is the one of Eq. 6 / Eq. 7 on the decoded
// weights, as in the im2col GEMM; only the order of the fp32 additions
// differs.
//
// One tcgen05.mma issuing thread sustains about one MMA per 27 ns, and
// every mbarrier wait placed between its issues costs it about 130 ns more
// (measured on GB300), while the tensor core needs ~25 ns for a
// 128 x 64 x 16 MMA.  So a tile's MMAs (taps x chunks x 4) run between
// waits on whole halo chunks, with slots and phases as running counters and
// the 3x3 taps unrolled, and two MMA warps take alternate tiles, each with
// its own halo ring and accumulators, so one warp's waits overlap the
// other's issues.
//
// Warp roles (one persistent CTA per SM): warp 0 issues the TMA loads, warps
// 1-2 the MMAs (M=128, N=BN, K=16, A and B from shared memory; warp 1 also
// allocates the TMEM), warps 3-6 read the accumulators, add bias /
// residual, apply the activation, convert to bf16 and write the valid rows
// into a staging tile laid out as the output rows, stored with one TMA box
// per output row.  Every wait is bounded.
#include "conv_common.cuh"
#include "conv_dispatch.h"
#include "tc_maps.h"
#include "tc_ptx.cuh"

#include <cuda.h>

#include <algorithm>
#include <mutex>
#include <type_traits>

namespace onexn {

namespace {

constexpr int kBM = 128;           // M rows per tile
constexpr int kRow = 128;          // bytes of K per shared-memory row (64 bf16)
constexpr int kBK = 64;            // channels per chunk
constexpr int kSmemMax = 232448;   // dynamic shared memory per CTA (opt-in maximum)
constexpr int kAccMax = 4;
constexpr int kMmaWarps = 2;
constexpr int kEpiWarp0 = 1 + kMmaWarps;
constexpr int kWarps = kEpiWarp0 + 4;
constexpr int kMaxHalo = 6;        // halo slots at most (all rings)
constexpr int kBarBytes = (2 * kMaxHalo + 1 + 2 * kAccMax + kMmaWarps) * 8;
constexpr double kMinRowFill = 0.85;   // valid share of the M rows below which the im2col form is kept

struct HaloPlan {
    int Wp, R, Rh, n_rb;           // padded width, output rows per tile, halo rows, row blocks per image
    int n_cc, n_taps, n_tn, n_m;   // chunks, taps, column tiles, pixel tiles (images x row blocks)
    int S_r, n_mma;                // halo slots per MMA warp, MMA warps
    int grid;                      // CTAs: a multiple of n_tn, CTA b serves column tile b % n_tn
    uint32_t halo_tx, slot_bytes, out_row_bytes, b_bytes;
    uint32_t off_halo, off_out, off_bias, off_bar, bytes;
    FastDiv div_rb;
};

constexpr int pow2_cols(int v, int p = 32) { return p >= v ? p : pow2_cols(v, 2 * p); }

template <int BN>
struct HaloTmem {
    static constexpr int kAccFit = 512 / BN;
    static constexpr int kAcc = kAccFit > kAccMax ? kAccMax : kAccFit;   // a multiple of kMmaWarps
    static constexpr int kCols = pow2_cols(kAcc * BN);
    static_assert(kAcc % kMmaWarps == 0, "accumulators per MMA warp");
};

__device__ __forceinline__ bool epi_all4(bool ok)
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

// KS = 3: 3x3 kernel, taps unrolled; KS = 0: any kernel shape.
template <int BN, int KS>
__global__ void __launch_bounds__(kWarps * 32, 1)
halo_conv_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_x,
                 const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_y,
                 const HaloPlan hp)
{
    using TM = HaloTmem<BN>;
    constexpr int kAcc = TM::kAcc;
    constexpr uint32_t kBTile = BN * kRow;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    const uint32_t sB = base;                       // the column tile's weights: (tap, chunk) B tiles
    const uint32_t sH = base + hp.off_halo;         // halo slots: ring j = slots j*S_r .. j*S_r + S_r - 1
    const uint32_t bar_hfull = base + hp.off_bar;
    const uint32_t bar_hempty = bar_hfull + 8 * kMaxHalo;
    const uint32_t bar_bfull = bar_hempty + 8 * kMaxHalo;
    const uint32_t bar_tfull = bar_bfull + 8;
    const uint32_t bar_tempty = bar_tfull + 8 * kAccMax;
    const uint32_t bar_drain = bar_tempty + 8 * kAccMax;   // one per MMA warp
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + hp.off_bar + kBarBytes);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < kMaxHalo; ++s) {
            mbar_init(bar_hfull + 8 * s, 1);
            mbar_init(bar_hempty + 8 * s, 1);
        }
        mbar_init(bar_bfull, 1);
        for (int b = 0; b < kAccMax; ++b) {
            mbar_init(bar_tfull + 8 * b, 1);
            mbar_init(bar_tempty + 8 * b, 128);
        }
        for (int j = 0; j < kMmaWarps; ++j) mbar_init(bar_drain + 8 * j, 1);
        fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(holder), TM::kCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;
    // a programmatic dependent of the previous kernel on the stream: global
    // memory is touched only after it has completed
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    auto abort_now = [&]() { atomicOr(a.status, kStatusTimeout); };
    // this CTA's column tile and pixel tiles: tm = m0, m0 + m_step, ...
    const int tn = static_cast<int>(blockIdx.x) % hp.n_tn;
    const int m0 = static_cast<int>(blockIdx.x) / hp.n_tn, m_step = hp.grid / hp.n_tn;

    if (warp == 0) {
        // ============================ producer ============================
        if (lane == 0) {
            bool failed = false;
            tc::mbar_arrive_expect_tx(bar_bfull, hp.b_bytes);
            for (int tap = 0, q = 0; tap < hp.n_taps; ++tap)
                for (int cc = 0; cc < hp.n_cc; ++cc, ++q)
                    tc::tma_load_2d(sB + q * kBTile, &tmap_w, tap * a.C + cc * kBK, tn * BN, bar_bfull);
            // per ring: loads issued so far (slot = count % S_r, phase = (count / S_r) & 1)
            int issued0 = 0, issued1 = 0;
            int si = 0;
            for (int tm = m0; tm < hp.n_m && !failed; tm += m_step, ++si) {
                const int j = hp.n_mma > 1 ? (si & 1) : 0;
                const int n = static_cast<int>(hp.div_rb.div(tm)), rb = tm - n * hp.n_rb;
                const int h0 = rb * hp.R;
                int cnt = j ? issued1 : issued0;
                for (int cc = 0; cc < hp.n_cc; ++cc, ++cnt) {
                    const int round = cnt / hp.S_r;
                    const int slot = j * hp.S_r + (cnt - round * hp.S_r);
                    if (round >= 1 && !mbar_wait(bar_hempty + 8 * slot, (round - 1) & 1)) {
                        abort_now(); failed = true; break;
                    }
                    tc::mbar_arrive_expect_tx(bar_hfull + 8 * slot, hp.halo_tx);
                    tc::tma_load_im2col_4d(sH + slot * hp.slot_bytes, &tmap_x, cc * kBK, -a.pw, h0 - a.ph, n, 0, 0,
                                           bar_hfull + 8 * slot);
                }
                if (j) issued1 = cnt; else issued0 = cnt;
            }
        }
        __syncwarp();
    } else if (warp < kEpiWarp0) {
        // ============================== MMA ==============================
        const int j = warp - 1;
        if (lane == 0 && j < hp.n_mma) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, BN);
            constexpr uint32_t kBDesc = BN * kRow / 16;          // descriptor units between B tiles
            bool failed = !mbar_wait(bar_bfull, 0);
            if (failed) abort_now();
            const uint64_t b_desc0 = tc::desc_kmajor_sw128(sB);
            const uint32_t row_step = static_cast<uint32_t>(a.dh * hp.Wp) * (kRow / 16);   // per kh, descriptor units
            const uint32_t col_step = static_cast<uint32_t>(a.dw) * (kRow / 16);           // per kw
            const uint32_t b_tap = static_cast<uint32_t>(hp.n_cc) * kBDesc;                 // per tap
            const int per = kAcc / hp.n_mma;        // accumulators of this warp: j, j + n_mma, ...
            int hs = 0, hph = 0, si = 0, k = 0;     // k: this warp's tile count
            for (int tm = m0; tm < hp.n_m && !failed; tm += m_step, ++si) {
                if (hp.n_mma > 1 && (si & 1) != j) continue;
                const int acc = j + hp.n_mma * (k % per), use = k / per;
                ++k;
                if (use >= 1 && !mbar_wait(bar_tempty + 8 * acc, (use - 1) & 1)) {
                    abort_now(); failed = true; break;
                }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + static_cast<uint32_t>(acc) * BN;
                for (int cc = 0; cc < hp.n_cc; ++cc) {
                    const int slot = j * hp.S_r + hs;
                    if (!mbar_wait(bar_hfull + 8 * slot, hph)) { abort_now(); failed = true; break; }
                    tc::fence_after_sync();
                    const uint64_t hd = tc::desc_kmajor_sw128(sH + static_cast<uint32_t>(slot) * hp.slot_bytes);
                    const uint64_t bd_cc = b_desc0 + static_cast<uint32_t>(cc) * kBDesc;
                    const uint32_t acc0 = cc != 0 ? 1u : 0u;
                    auto tap_mmas = [&](uint64_t ad, uint64_t bd, uint32_t first_acc) {
                        tc::mma_bf16(d_tmem, ad, bd, idesc, first_acc);
#pragma unroll
                        for (int kk = 1; kk < kBK / 16; ++kk) tc::mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, idesc, 1u);
                    };
                    if constexpr (KS > 0) {
#pragma unroll
                        for (int tap = 0; tap < KS * KS; ++tap)
                            tap_mmas(hd + (tap / KS) * row_step + (tap % KS) * col_step, bd_cc + tap * b_tap,
                                     tap == 0 ? acc0 : 1u);
                    } else {
                        int kw = 0, kh = 0;
                        for (int tap = 0; tap < hp.n_taps; ++tap) {
                            tap_mmas(hd + kh * row_step + kw * col_step, bd_cc + static_cast<uint32_t>(tap) * b_tap,
                                     tap == 0 ? acc0 : 1u);
                            if (++kw == a.KW) { kw = 0; ++kh; }
                        }
                    }
                    tc::commit(bar_hempty + 8 * slot);
                    if (++hs == hp.S_r) { hs = 0; hph ^= 1; }
                }
                if (failed) break;
                tc::commit(bar_tfull + 8 * acc);
            }
            tc::commit(bar_drain + 8 * j);
            if (!mbar_wait(bar_drain + 8 * j, 0)) abort_now();
        }
        __syncwarp();
    } else {
        // ============================ epilogue ============================
        // Thread (warp w, lane i) owns TMEM lane m = 32*(w%4) + i, output
        // pixel (h0 + m / Wp, m % Wp) of the tile.  Per 64-column atom: read
        // the accumulator, add bias (and residual), activate, convert, write
        // the 128-byte row into the staging tile of its output row (double
        // buffered across atoms), then one thread stores each output row.
        auto epilogue = [&](auto res_c, auto act_c) {
            constexpr bool kRes = decltype(res_c)::value;
            constexpr int kAct = decltype(act_c)::value;
            constexpr int kAtoms = BN / 64;
            const int q = warp & 3;
            const int m = 32 * q + lane;
            const int mr = m / hp.Wp, mw = m - mr * hp.Wp;
            const bool leader = (warp == kEpiWarp0) && lane == 0;
            const uint32_t sout = base + hp.off_out;
            const uint32_t buf_bytes = static_cast<uint32_t>(hp.R) * hp.out_row_bytes;
            float *sbias = reinterpret_cast<float *>(smem + hp.off_bias);
            const float4 *sb4 = reinterpret_cast<const float4 *>(sbias);
            for (int c = m; c < BN; c += 128) {      // the column tile's bias, once
                const int o = tn * BN + c;
                sbias[c] = (a.bias && o < a.C_out) ? __ldg(a.bias + o) : 0.f;
            }
            tc::named_bar(1, 128);
            // accumulator of the CTA's tile si: MMA warp j = si % n_mma uses
            // j, j + n_mma, ... in turn
            const int per = kAcc / hp.n_mma;
            int n_emit = 0, si = 0;
            for (int tm = m0; tm < hp.n_m; tm += m_step, ++si) {
                const int j = hp.n_mma > 1 ? (si & 1) : 0;
                const int kj = hp.n_mma > 1 ? (si >> 1) : si;          // MMA warp j's tile count before this one
                const int acc = j + hp.n_mma * (kj % per), use = kj / per;
                if (!epi_all4(mbar_wait(bar_tfull + 8 * acc, use & 1))) { abort_now(); break; }
                tc::fence_after_sync();
                const int n = static_cast<int>(hp.div_rb.div(tm)), rb = tm - n * hp.n_rb;
                const int h0 = rb * hp.R;
                const int R_t = min(hp.R, a.Ho - h0);
                const bool valid = mr < R_t && mw < a.Wo;
                const int64_t pix = (static_cast<int64_t>(n) * a.Ho + h0 + mr) * a.Wo + mw;
                const uint32_t t_acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + acc * BN;
#pragma unroll 1
                for (int at = 0; at < kAtoms; ++at) {
                    const int col0 = tn * BN + at * 64;
                    uint32_t r0[32], r1[32];
                    tc::ld_32x32b_x32(t_acc + at * 64, r0);
                    tc::ld_32x32b_x32(t_acc + at * 64 + 32, r1);
                    tc::ld_wait();
                    if (at == kAtoms - 1) {
                        tc::fence_before_sync();
                        mbar_arrive(bar_tempty + 8 * acc);
                    }
                    if (col0 >= a.C_out) continue;   // uniform: the atom lies past y's columns
                    const uint32_t buf = sout + static_cast<uint32_t>(n_emit & 1) * buf_bytes;
                    ++n_emit;
                    // the stores of two atoms back have read this buffer
                    if (leader) tc::bulk_wait_read1();
                    tc::named_bar(1, 128);
                    if (valid) {
                        const uint4 *res = nullptr;
                        if constexpr (kRes)
                            res = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(a.residual) +
                                                                  pix * a.C_out + col0);
                        const uint32_t dst = buf + static_cast<uint32_t>(mr) * hp.out_row_bytes +
                                             static_cast<uint32_t>(mw) * kRow;
#pragma unroll
                        for (int jj = 0; jj < 8; ++jj) {          // 16-byte chunk jj: columns 8jj .. 8jj+7
                            uint32_t rw[4] = {0u, 0u, 0u, 0u};
                            if constexpr (kRes) {
                                if (col0 + 8 * jj < a.C_out) {
                                    const uint4 rv = __ldg(res + jj);
                                    rw[0] = rv.x; rw[1] = rv.y; rw[2] = rv.z; rw[3] = rv.w;
                                }
                            }
                            const float4 b0 = sb4[at * 16 + 2 * jj], b1 = sb4[at * 16 + 2 * jj + 1];
                            const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
                            uint32_t w[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const int c = 8 * jj + 2 * e;
                                const uint32_t u0 = c < 32 ? r0[c] : r1[c - 32];
                                const uint32_t u1 = c + 1 < 32 ? r0[c + 1] : r1[c + 1 - 32];
                                float v0 = __uint_as_float(u0) + bb[2 * e], v1 = __uint_as_float(u1) + bb[2 * e + 1];
                                if constexpr (kRes) {
                                    v0 += bf16lo(rw[e]);
                                    v1 += bf16hi(rw[e]);
                                }
                                w[e] = pack_bf16x2(activate_c<kAct>(v0), activate_c<kAct>(v1));
                            }
                            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(
                                             dst + ((jj ^ (mw & 7)) << 4)),
                                         "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                                         : "memory");
                        }
                    }
                    tc::fence_proxy_async_smem();
                    tc::named_bar(1, 128);
                    if (leader) {
                        for (int r = 0; r < R_t; ++r)
                            tc::tma_store_3d(&tmap_y, col0, 0, n * a.Ho + h0 + r,
                                             buf + static_cast<uint32_t>(r) * hp.out_row_bytes);
                        tc::bulk_commit();
                    }
                }
            }
            if (leader) tc::bulk_wait0();
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
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, TM::kCols);
    }
}

// ---------------------------------------------------------------------------
// Streamed-weights form (layers whose column tile of weights does not fit in
// shared memory next to the halo slots, and strided layers).  The output of
// an image is laid out in the padded space of Hp rows of Wp positions
// (position (n*Hp + r)*Wp + w is output pixel (n, r, w) when r < Ho and
// w < Wo, else a dropped row).  For stride 1 the input is in the same
// space (row r, column w = input pixel (r - ph, w - pw)), Hp = Ho + (KH-1)*dh,
// Wp = Wo + (KW-1)*dw, and output position P of tap (kh, kw) reads input
// position P + kh*dh*Wp + kw*dw.  A strided layer is split into the phases
// of its input (the pixels s*i + phase, per dimension): tap k reads phase
// (k*d - p) mod s at an index shifted by floor((k*d - p) / s), so each phase
// is a stride-1 problem on its own padded space of the same Hp x Wp, and
// each tap a shift within one phase (phase_dim below).  A tile is 256
// consecutive positions, two M = 128 halves; it may run across rows and
// images, so only the padding positions are wasted.  Per (64-channel chunk,
// phase) one TMA im2col load, stepping by the layer's strides and offset by
// the phase, brings the tile's positions plus the largest shift (the
// traversal continues into the next image, zeros after the last one), and
// the A operand of (half h, tap) is that buffer viewed from row 128*h +
// the tap's shift.  The weights are streamed: one B stage holds one kernel
// row of taps (stride-1 3x3) or one tap, 128-byte swizzled, shared by both
// halves.  MMA warp h issues the MMAs of half h (its own accumulators), so
// each issuing thread meets one stage wait per stage; the epilogue warps
// (two per TMEM lane quarter, one per half) store their valid rows straight
// to global memory.
constexpr int kWRows = 2 * kBM;            // positions per tile
constexpr int kWEpiWarp0 = 3;
constexpr int kWWarps = kWEpiWarp0 + 8;    // producer, two MMA warps, eight epilogue warps
constexpr int kWMaxHalo = 4;
constexpr int kWMaxStages = 12;
constexpr int kWMaxTaps = 49;              // taps of the tap table (7x7 at most)
constexpr int kWMaxPhases = 4;
constexpr int kWAccMax = 4;
constexpr int kWBarBytes = (2 * kWMaxHalo + 2 * kWMaxStages + 4 * kWAccMax + 2) * 8;

struct WidePlan {
    int Wp, Hp;                    // padded output width and rows per image
    int n_cc, n_taps, tps, n_st;   // chunks, taps, taps per B stage, B stages per chunk
    int n_tn, n_m, grid;           // column tiles, position tiles, CTAs (a multiple of n_tn)
    int S_h, S_b;                  // halo slots, B stages
    int n_ph;                      // input phases (1 for stride 1)
    int lower_w, lower_h;          // TMA start of padded position (r, c): (lower_w + sw*c, lower_h + sh*r)
    uint32_t halo_pix, halo_tx, slot_bytes, stage_bytes;
    uint32_t off_b, off_bias, off_bar, off_tab, bytes;
    FastDiv div_img, div_wp;       // Hp*Wp, Wp
    // tap table (grouped by phase): K tap index << 16 | A view shift in rows;
    // phase table: first tap | end tap << 8 | im2col w offset << 16 | h offset << 24
    uint32_t tap[kWMaxTaps];
    uint32_t ph[kWMaxPhases];
};

template <int BN>
struct WideTmem {
    static constexpr int kAccFit = 512 / (2 * BN);
    static constexpr int kAcc = kAccFit > kWAccMax ? kWAccMax : kAccFit;   // buffers of two halves
    static constexpr int kCols = pow2_cols(kAcc * 2 * BN);
};

// KS = 3: stride-1 3x3 kernel (a B stage is one kernel row of three taps,
// unrolled); KS = 0: any kernel shape and stride, one halo per (chunk,
// phase) and one tap per stage, from the plan's tap table.
template <int BN, int KS>
__global__ void __launch_bounds__(kWWarps * 32, 1)
halo_wide_kernel(const ConvArgs a, const __grid_constant__ CUtensorMap tmap_x,
                 const __grid_constant__ CUtensorMap tmap_w, const WidePlan wp)
{
    using TM = WideTmem<BN>;
    constexpr int kAcc = TM::kAcc;
    constexpr uint32_t kBTile = BN * kRow;
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *smem = smem_raw + (base - raw);
    const uint32_t sH = base;                      // halo slots
    const uint32_t sB = base + wp.off_b;           // B stages
    const uint32_t bar_hfull = base + wp.off_bar;
    const uint32_t bar_hempty = bar_hfull + 8 * kWMaxHalo;
    const uint32_t bar_bfull = bar_hempty + 8 * kWMaxHalo;
    const uint32_t bar_bempty = bar_bfull + 8 * kWMaxStages;
    const uint32_t bar_tfull = bar_bempty + 8 * kWMaxStages;   // [acc][half]
    const uint32_t bar_tempty = bar_tfull + 16 * kWAccMax;     // [acc][half]
    const uint32_t bar_drain = bar_tempty + 16 * kWAccMax;     // one per MMA warp
    uint32_t *holder = reinterpret_cast<uint32_t *>(smem + wp.off_bar + kWBarBytes);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        for (int s = 0; s < kWMaxHalo; ++s) {
            mbar_init(bar_hfull + 8 * s, 1);
            mbar_init(bar_hempty + 8 * s, 2);       // both MMA warps commit
        }
        for (int s = 0; s < kWMaxStages; ++s) {
            mbar_init(bar_bfull + 8 * s, 1);
            mbar_init(bar_bempty + 8 * s, 2);
        }
        for (int b = 0; b < 2 * kWAccMax; ++b) {
            mbar_init(bar_tfull + 8 * b, 1);
            mbar_init(bar_tempty + 8 * b, 128);     // the four epilogue warps of the half
        }
        for (int j = 0; j < 2; ++j) mbar_init(bar_drain + 8 * j, 1);
        fence_mbar_init();
        uint32_t *tab = reinterpret_cast<uint32_t *>(smem + wp.off_tab);
        for (int i = 0; i < kWMaxTaps; ++i) tab[i] = wp.tap[i];
        for (int i = 0; i < kWMaxPhases; ++i) tab[kWMaxTaps + i] = wp.ph[i];
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(holder), TM::kCols);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *holder;
    // a programmatic dependent of the previous kernel on the stream: global
    // memory is touched only after it has completed
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    auto abort_now = [&]() { atomicOr(a.status, kStatusTimeout); };
    const int tn = static_cast<int>(blockIdx.x) % wp.n_tn;
    const int m0 = static_cast<int>(blockIdx.x) / wp.n_tn, m_step = wp.grid / wp.n_tn;
    const uint32_t img = static_cast<uint32_t>(wp.Hp) * static_cast<uint32_t>(wp.Wp);
    const uint32_t *s_tap = reinterpret_cast<const uint32_t *>(smem + wp.off_tab);
    const uint32_t *s_ph = s_tap + kWMaxTaps;
    // phases and their B stages: the stride-1 3x3 form has one phase of
    // n_st stages (kernel rows); the general one takes both from the tables
    const int n_ph = KS > 0 ? 1 : wp.n_ph;
    auto ph_stages = [&](int ph, int &st0, int &st1) {
        if constexpr (KS > 0) {
            st0 = 0;
            st1 = wp.n_st;
        } else {
            st0 = static_cast<int>(s_ph[ph] & 0xffu);
            st1 = static_cast<int>((s_ph[ph] >> 8) & 0xffu);
        }
    };

    if (warp == 0) {
        // ============================ producer ============================
        if (lane == 0) {
            bool failed = false;
            int hs = 0, hround = 0, bs = 0, bround = 0;
            for (int tm = m0; tm < wp.n_m && !failed; tm += m_step) {
                const uint32_t P0 = static_cast<uint32_t>(tm) * kWRows;
                const uint32_t n0 = wp.div_img.div(P0), rem = P0 - n0 * img;
                const uint32_t r0 = wp.div_wp.div(rem), w0 = rem - r0 * static_cast<uint32_t>(wp.Wp);
                const int w_start = wp.lower_w + a.sw * static_cast<int>(w0);
                const int h_start = wp.lower_h + a.sh * static_cast<int>(r0);
                for (int u = 0; u < wp.n_cc * n_ph && !failed; ++u) {
                    const int cc = u / n_ph, ph = u - cc * n_ph;
                    if (hround >= 1 && !mbar_wait(bar_hempty + 8 * hs, (hround - 1) & 1)) {
                        failed = true;
                        break;
                    }
                    const uint32_t phv = KS > 0 ? 0u : s_ph[ph];
                    tc::mbar_arrive_expect_tx(bar_hfull + 8 * hs, wp.halo_tx);
                    tc::tma_load_im2col_4d(sH + static_cast<uint32_t>(hs) * wp.slot_bytes, &tmap_x, cc * kBK,
                                           w_start, h_start, static_cast<int>(n0),
                                           static_cast<uint16_t>((phv >> 16) & 0xffu),
                                           static_cast<uint16_t>(phv >> 24), bar_hfull + 8 * hs);
                    if (++hs == wp.S_h) { hs = 0; ++hround; }
                    int st0, st1;
                    ph_stages(ph, st0, st1);
                    for (int st = st0; st < st1; ++st) {
                        if (bround >= 1 && !mbar_wait(bar_bempty + 8 * bs, (bround - 1) & 1)) {
                            failed = true;
                            break;
                        }
                        tc::mbar_arrive_expect_tx(bar_bfull + 8 * bs, wp.stage_bytes);
                        const uint32_t dst = sB + static_cast<uint32_t>(bs) * wp.stage_bytes;
                        for (int i = 0; i < wp.tps; ++i) {
                            const int ktap = KS > 0 ? st * wp.tps + i : static_cast<int>(s_tap[st] >> 16);
                            tc::tma_load_2d(dst + static_cast<uint32_t>(i) * kBTile, &tmap_w,
                                            ktap * a.C + cc * kBK, tn * BN, bar_bfull + 8 * bs);
                        }
                        if (++bs == wp.S_b) { bs = 0; ++bround; }
                    }
                }
            }
            if (failed) abort_now();
        }
        __syncwarp();
    } else if (warp < kWEpiWarp0) {
        // ============================== MMA ==============================
        const int h = warp - 1;                    // the half this warp multiplies
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_bf16_f32(kBM, BN);
            constexpr uint32_t kBDesc = kBTile / 16;                  // descriptor units between B tiles
            const uint32_t row_step = static_cast<uint32_t>(a.dh * wp.Wp) * (kRow / 16);   // per kh
            const uint32_t col_step = static_cast<uint32_t>(a.dw) * (kRow / 16);           // per kw
            const uint32_t half_off = static_cast<uint32_t>(h * kBM) * (kRow / 16);
            bool failed = false;
            int hs = 0, hph = 0, bs = 0, bph = 0, k = 0;
            for (int tm = m0; tm < wp.n_m && !failed; tm += m_step, ++k) {
                const int acc = k % kAcc, use = k / kAcc;
                if (use >= 1 && !mbar_wait(bar_tempty + 8 * (2 * acc + h), (use - 1) & 1)) {
                    failed = true;
                    break;
                }
                tc::fence_after_sync();
                const uint32_t d_tmem = tmem + static_cast<uint32_t>(2 * acc + h) * BN;
                for (int u = 0; u < wp.n_cc * n_ph && !failed; ++u) {
                    const int cc = u / n_ph, ph = u - cc * n_ph;
                    if (!mbar_wait(bar_hfull + 8 * hs, hph)) { failed = true; break; }
                    tc::fence_after_sync();
                    const uint64_t hd = tc::desc_kmajor_sw128(sH + static_cast<uint32_t>(hs) * wp.slot_bytes) + half_off;
                    int st0, st1;
                    ph_stages(ph, st0, st1);
                    for (int st = st0; st < st1; ++st) {
                        if (!mbar_wait(bar_bfull + 8 * bs, bph)) { failed = true; break; }
                        tc::fence_after_sync();
                        const uint64_t bd = tc::desc_kmajor_sw128(sB + static_cast<uint32_t>(bs) * wp.stage_bytes);
                        const uint32_t first = (cc == 0 && st == 0) ? 0u : 1u;
                        auto tap_mmas = [&](uint64_t ad, uint64_t b, uint32_t first_acc) {
                            tc::mma_bf16(d_tmem, ad, b, idesc, first_acc);
#pragma unroll
                            for (int kk = 1; kk < kBK / 16; ++kk) tc::mma_bf16(d_tmem, ad + 2 * kk, b + 2 * kk, idesc, 1u);
                        };
                        if constexpr (KS > 0) {
                            const uint64_t ad_row = hd + static_cast<uint32_t>(st) * row_step;
#pragma unroll
                            for (int t = 0; t < KS; ++t)
                                tap_mmas(ad_row + t * col_step, bd + t * kBDesc, t == 0 ? first : 1u);
                        } else {
                            tap_mmas(hd + (s_tap[st] & 0xffffu) * (kRow / 16), bd, first);
                        }
                        tc::commit(bar_bempty + 8 * bs);
                        if (++bs == wp.S_b) { bs = 0; bph ^= 1; }
                    }
                    if (failed) break;
                    tc::commit(bar_hempty + 8 * hs);
                    if (++hs == wp.S_h) { hs = 0; hph ^= 1; }
                }
                if (failed) break;
                tc::commit(bar_tfull + 8 * (2 * acc + h));
            }
            if (failed) abort_now();
            // everything this thread issued completes before the TMEM is freed
            tc::commit(bar_drain + 8 * h);
            if (!mbar_wait(bar_drain + 8 * h, 0)) abort_now();
        }
        __syncwarp();
    } else {
        // ============================ epilogue ============================
        // Warp w (3..10) reads TMEM lane quarter w % 4 of half (w - 3) / 4:
        // thread (w, i) owns position 128*half + 32*(w % 4) + i of each tile.
        // Per 64-column atom: read the accumulator, add bias (and
        // residual), activate, convert to bf16 and store the pixel's 128
        // bytes when the position is an output pixel.
        auto epilogue = [&](auto res_c, auto act_c) {
            constexpr bool kRes = decltype(res_c)::value;
            constexpr int kAct = decltype(act_c)::value;
            constexpr int kAtoms = BN / 64;
            const int h = (warp - kWEpiWarp0) >> 2, q = warp & 3;
            const int m = h * kBM + 32 * q + lane;
            float *sbias = reinterpret_cast<float *>(smem + wp.off_bias);
            const float4 *sb4 = reinterpret_cast<const float4 *>(sbias);
            for (int c = tid - kWEpiWarp0 * 32; c < BN; c += 256) {     // the column tile's bias, once
                const int o = tn * BN + c;
                sbias[c] = (a.bias && o < a.C_out) ? __ldg(a.bias + o) : 0.f;
            }
            tc::named_bar(1, 256);
            __nv_bfloat16 *y = static_cast<__nv_bfloat16 *>(a.y);
            int k = 0;
            for (int tm = m0; tm < wp.n_m; tm += m_step, ++k) {
                const int acc = k % kAcc, use = k / kAcc;
                if (!mbar_wait(bar_tfull + 8 * (2 * acc + h), use & 1)) { abort_now(); break; }
                tc::fence_after_sync();
                const uint32_t P = static_cast<uint32_t>(tm) * kWRows + static_cast<uint32_t>(m);
                const uint32_t n = wp.div_img.div(P), rem = P - n * img;
                const uint32_t r = wp.div_wp.div(rem), w = rem - r * static_cast<uint32_t>(wp.Wp);
                const bool valid = static_cast<int>(n) < a.B && static_cast<int>(r) < a.Ho && static_cast<int>(w) < a.Wo;
                const int64_t pix = (static_cast<int64_t>(n) * a.Ho + r) * a.Wo + w;
                const uint32_t t_acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(2 * acc + h) * BN;
#pragma unroll 1
                for (int at = 0; at < kAtoms; ++at) {
                    const int col0 = tn * BN + at * 64;
                    uint32_t r0[32], r1[32];
                    tc::ld_32x32b_x32(t_acc + at * 64, r0);
                    tc::ld_32x32b_x32(t_acc + at * 64 + 32, r1);
                    tc::ld_wait();
                    if (at == kAtoms - 1) {
                        tc::fence_before_sync();
                        mbar_arrive(bar_tempty + 8 * (2 * acc + h));
                    }
                    if (!valid || col0 >= a.C_out) continue;
                    __nv_bfloat16 *yp = y + pix * a.C_out + col0;
                    const uint4 *res = nullptr;
                    if constexpr (kRes)
                        res = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(a.residual) +
                                                              pix * a.C_out + col0);
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj) {          // 16-byte chunk jj: columns 8jj .. 8jj+7
                        if (col0 + 8 * jj >= a.C_out) break;
                        uint32_t rw[4] = {0u, 0u, 0u, 0u};
                        if constexpr (kRes) {
                            const uint4 rv = __ldg(res + jj);
                            rw[0] = rv.x; rw[1] = rv.y; rw[2] = rv.z; rw[3] = rv.w;
                        }
                        const float4 b0 = sb4[at * 16 + 2 * jj], b1 = sb4[at * 16 + 2 * jj + 1];
                        const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
                        uint32_t wv[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int c = 8 * jj + 2 * e;
                            const uint32_t u0 = c < 32 ? r0[c] : r1[c - 32];
                            const uint32_t u1 = c + 1 < 32 ? r0[c + 1] : r1[c + 1 - 32];
                            float v0 = __uint_as_float(u0) + bb[2 * e], v1 = __uint_as_float(u1) + bb[2 * e + 1];
                            if constexpr (kRes) {
                                v0 += bf16lo(rw[e]);
                                v1 += bf16hi(rw[e]);
                            }
                            wv[e] = pack_bf16x2(activate_c<kAct>(v0), activate_c<kAct>(v1));
                        }
                        *reinterpret_cast<uint4 *>(yp + 8 * jj) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                    }
                }
            }
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
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, TM::kCols);
    }
}

uint32_t round1024(uint64_t v) { return static_cast<uint32_t>((v + 1023) & ~static_cast<uint64_t>(1023)); }

// The halo plan of a bf16 layer, or false when the layer keeps the im2col
// form: strided or 1x1 layers, rows too wide for one M tile, too many
// dropped M rows, or a column tile whose weights do not fit in shared
// memory next to two halo slots.  The column tile is the widest of 256 /
// 128 / 64 that fits (no wider than the output channels need).
bool halo_plan(const ConvArgs &a, int sms, HaloPlan *out, int *bn_out)
{
    if (a.sh != 1 || a.sw != 1 || a.KH * a.KW == 1 || a.Ho <= 0 || a.Wo <= 0 || a.B <= 0) return false;
    HaloPlan p{};
    p.Wp = a.Wo + (a.KW - 1) * a.dw;
    if (p.Wp > kBM) return false;
    p.R = std::min(kBM / p.Wp, a.Ho);
    p.n_rb = (a.Ho + p.R - 1) / p.R;
    const double fill = static_cast<double>(a.Ho) * a.Wo / (static_cast<double>(p.n_rb) * kBM);
    if (fill < kMinRowFill) return false;
    p.Rh = p.R + (a.KH - 1) * a.dh;
    if (p.Wp * p.Rh > 1024) return false;                 // positions per im2col load
    const int reach = (a.KH - 1) * a.dh * p.Wp + (a.KW - 1) * a.dw + kBM;   // rows an MMA view can read
    p.slot_bytes = round1024(static_cast<uint64_t>(std::max(p.Rh * p.Wp, reach)) * kRow);
    p.halo_tx = static_cast<uint32_t>(p.Wp * p.Rh * kRow);
    p.out_row_bytes = round1024(static_cast<uint64_t>(a.Wo) * kRow);
    p.n_cc = (a.C + kBK - 1) / kBK;
    p.n_taps = a.KH * a.KW;
    p.n_m = a.B * p.n_rb;
    const uint32_t staging = 2u * static_cast<uint32_t>(p.R) * p.out_row_bytes;
    int bn = 0;
    for (int cand : {256, 128, 64}) {
        if (cand > 64 && a.C_out <= cand / 2) continue;
        const uint64_t b_bytes = static_cast<uint64_t>(p.n_taps) * p.n_cc * cand * kRow;
        const uint64_t fixed = staging + round1024(static_cast<uint64_t>(cand) * 4 + kBarBytes + 16) + 1024;
        if (round1024(b_bytes) + 2ull * p.slot_bytes + fixed <= static_cast<uint64_t>(kSmemMax)) {
            bn = cand;
            p.b_bytes = static_cast<uint32_t>(b_bytes);
            const uint64_t left = kSmemMax - fixed - round1024(b_bytes);
            const int slots = static_cast<int>(std::min<uint64_t>(kMaxHalo, left / p.slot_bytes));
            // two MMA warps when each can keep two halo slots in flight
            p.n_mma = slots >= 2 * kMmaWarps ? kMmaWarps : 1;
            p.S_r = slots / p.n_mma;
            break;
        }
    }
    if (bn == 0) return false;
    p.n_tn = (a.C_out + bn - 1) / bn;
    if (p.n_tn > sms) return false;
    const int64_t tiles = static_cast<int64_t>(p.n_m) * p.n_tn;
    p.grid = static_cast<int>(std::min<int64_t>(tiles, sms) / p.n_tn * p.n_tn);
    p.off_halo = round1024(p.b_bytes);
    p.off_out = p.off_halo + static_cast<uint32_t>(p.S_r * p.n_mma) * p.slot_bytes;
    p.off_bias = p.off_out + staging;
    p.off_bar = p.off_bias + static_cast<uint32_t>(bn) * 4;
    p.bytes = p.off_bar + kBarBytes + 16;
    if (p.bytes + 1024 > static_cast<uint32_t>(kSmemMax)) return false;
    p.div_rb = FastDiv(static_cast<uint32_t>(p.n_rb));
    *out = p;
    *bn_out = bn;
    return true;
}

// im2col tensor map of the halo.  The traversal's bounding box is the
// padded image (corners innermost first: W, H): base positions lower ..
// W - 1 + upper, stepped by the traversal strides (the layer's strides for
// the streamed form, 1 for the resident one), each loading x at base + the
// load's im2col offsets (a phase of a strided layer, else 0).  So a load of
// `pixels` positions walks whole padded rows from its start, and one that
// runs past the padded image continues into the next image's rows (or zeros
// after the last image); those rows feed only dropped M rows.
bool box_ok(const int lower[2], const int upper[2])
{
    for (int i = 0; i < 2; ++i)
        if (lower[i] < -128 || lower[i] > 127 || upper[i] < -128 || upper[i] > 127) return false;
    return true;
}

bool halo_x_tmap(const ConvArgs &a, const int lower[2], const int upper[2], int estr_w, int estr_h, int pixels,
                 CUtensorMap *m)
{
    auto enc = encode_im2col_fn_public();
    if (!enc) return false;
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(a.C), static_cast<cuuint64_t>(a.W),
                                static_cast<cuuint64_t>(a.H), static_cast<cuuint64_t>(a.B)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(a.C) * 2, static_cast<cuuint64_t>(a.C) * 2 * a.W,
                                   static_cast<cuuint64_t>(a.C) * 2 * a.W * a.H};
    if (!box_ok(lower, upper)) return false;
    const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(estr_w), static_cast<cuuint32_t>(estr_h), 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(a.x), dims, strides, lower, upper, kBK,
               static_cast<cuuint32_t>(pixels), estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One spatial dimension of a (possibly strided) layer in the streamed form.
// Output o of tap k reads input s*o + q, q = k*d - p, which is phase
// q mod s of the input (the inputs s*i + phase) at phase index
// o + floor(q / s).  In the padded space, position c of a row holds phase
// index c + lo (lo = the smallest floor(q / s)), so tap k is a shift of
// floor(q / s) - lo positions, and the row is P = Out + (largest - smallest
// floor) long; the TMA traversal's base positions are s*(c + lo), i.e.
// lower = s*lo, and lower + s*(P - 1) is the last one (upper corner).
struct PhaseDim {
    int lo, P, lower;
    int phase[kWMaxTaps], shift[kWMaxTaps];
};

bool phase_dim(int K, int s, int p, int d, int Out, PhaseDim *g)
{
    if (K > kWMaxTaps || s < 1) return false;
    int lo = INT32_MAX, hi = INT32_MIN;
    for (int k = 0; k < K; ++k) {
        const int q = k * d - p;
        const int ph = ((q % s) + s) % s;
        g->phase[k] = ph;
        g->shift[k] = (q - ph) / s;
        lo = std::min(lo, g->shift[k]);
        hi = std::max(hi, g->shift[k]);
    }
    for (int k = 0; k < K; ++k) g->shift[k] -= lo;
    g->lo = lo;
    g->P = Out + (hi - lo);
    g->lower = s * lo;
    return true;
}

// The streamed-weights plan, or false: 1x1 layers, too many dropped
// positions (Ho*Wo below 85% of Hp*Wp), more than four input phases
// (strides above 2 in both dimensions) or 49 taps, more positions per load
// than one im2col load can walk, a traversal box out of the TMA's range, or
// shared memory for fewer than two B stages.  The column tile is 128 (64
// when the output channels fit in 64), so that two accumulator buffers of
// two halves fit in the TMEM.
bool wide_plan(const ConvArgs &a, int sms, WidePlan *out, int *bn_out)
{
    if (a.KH * a.KW == 1 || a.Ho <= 0 || a.Wo <= 0 || a.B <= 0 || a.KH * a.KW > kWMaxTaps) return false;
    WidePlan p{};
    PhaseDim gw, gh;
    if (!phase_dim(a.KW, a.sw, a.pw, a.dw, a.Wo, &gw) || !phase_dim(a.KH, a.sh, a.ph, a.dh, a.Ho, &gh)) return false;
    p.Wp = gw.P;
    p.Hp = gh.P;
    p.lower_w = gw.lower;
    p.lower_h = gh.lower;
    const int lower[2] = {p.lower_w, p.lower_h};
    const int upper[2] = {p.lower_w + a.sw * (p.Wp - 1) - (a.W - 1), p.lower_h + a.sh * (p.Hp - 1) - (a.H - 1)};
    if (!box_ok(lower, upper)) return false;
    const double fill = static_cast<double>(a.Ho) * a.Wo / (static_cast<double>(p.Hp) * p.Wp);
    if (fill < kMinRowFill) return false;
    const int64_t positions = static_cast<int64_t>(a.B) * p.Hp * p.Wp;
    if (positions + kWRows > INT32_MAX) return false;
    // the tap table grouped by input phase (phases in order of first use)
    int ph_key[kWMaxPhases], n_ph = 0, t = 0, max_shift = 0;
    for (int kh = 0; kh < a.KH; ++kh)
        for (int kw = 0; kw < a.KW; ++kw) {
            const int key = gh.phase[kh] * 256 + gw.phase[kw];
            int i = 0;
            while (i < n_ph && ph_key[i] != key) ++i;
            if (i == n_ph) {
                if (n_ph == kWMaxPhases) return false;
                ph_key[n_ph++] = key;
            }
        }
    for (int i = 0; i < n_ph; ++i) {
        const int t0 = t;
        for (int kh = 0; kh < a.KH; ++kh)
            for (int kw = 0; kw < a.KW; ++kw) {
                if (gh.phase[kh] * 256 + gw.phase[kw] != ph_key[i]) continue;
                const int shift = gh.shift[kh] * p.Wp + gw.shift[kw];
                max_shift = std::max(max_shift, shift);
                if (shift > 0xffff) return false;
                p.tap[t++] = (static_cast<uint32_t>(kh * a.KW + kw) << 16) | static_cast<uint32_t>(shift);
            }
        p.ph[i] = static_cast<uint32_t>(t0) | (static_cast<uint32_t>(t) << 8) |
                  (static_cast<uint32_t>(ph_key[i] & 0xff) << 16) | (static_cast<uint32_t>(ph_key[i] >> 8) << 24);
    }
    p.n_ph = n_ph;
    const int64_t halo = kWRows + max_shift;
    if (halo > 1024) return false;                        // positions per im2col load
    p.halo_pix = static_cast<uint32_t>(halo);
    p.halo_tx = p.halo_pix * kRow;
    p.slot_bytes = round1024(static_cast<uint64_t>(p.halo_pix) * kRow);
    p.n_cc = (a.C + kBK - 1) / kBK;
    p.n_taps = a.KH * a.KW;
    // stride-1 3x3: one phase, B stages of one kernel row (the unrolled form)
    const bool k3 = a.KH == 3 && a.KW == 3 && a.sh == 1 && a.sw == 1;
    p.tps = k3 ? 3 : 1;
    p.n_st = p.n_taps / p.tps;
    const int bn = a.C_out <= 64 ? 64 : 128;
    p.stage_bytes = static_cast<uint32_t>(p.tps * bn * kRow);
    const uint64_t tab = (kWMaxTaps + kWMaxPhases) * 4;
    const uint64_t fixed = static_cast<uint64_t>(bn) * 4 + kWBarBytes + 16 + tab + 1024;   // + base alignment
    // halo slots: two for one phase; with several phases (each read by
    // fewer taps) up to four, keeping at least four B stages
    int S_h = n_ph > 1 ? kWMaxHalo : 2;
    while (S_h > 2 && static_cast<uint64_t>(S_h) * p.slot_bytes + fixed + 4ull * p.stage_bytes >
                          static_cast<uint64_t>(kSmemMax))
        --S_h;
    p.S_h = S_h;
    const uint64_t halo_bytes = static_cast<uint64_t>(p.S_h) * p.slot_bytes;
    if (halo_bytes + fixed + 2ull * p.stage_bytes > static_cast<uint64_t>(kSmemMax)) return false;
    p.S_b = static_cast<int>(std::min<uint64_t>(kWMaxStages, (kSmemMax - fixed - halo_bytes) / p.stage_bytes));
    p.n_tn = (a.C_out + bn - 1) / bn;
    if (p.n_tn > sms) return false;
    p.n_m = static_cast<int>((positions + kWRows - 1) / kWRows);
    const int64_t tiles = static_cast<int64_t>(p.n_m) * p.n_tn;
    p.grid = static_cast<int>(std::min<int64_t>(tiles, sms) / p.n_tn * p.n_tn);
    p.off_b = static_cast<uint32_t>(halo_bytes);
    p.off_bias = p.off_b + static_cast<uint32_t>(p.S_b) * p.stage_bytes;
    p.off_bar = p.off_bias + static_cast<uint32_t>(bn) * 4;
    p.off_tab = p.off_bar + kWBarBytes + 16;
    p.bytes = p.off_tab + static_cast<uint32_t>(tab);
    if (p.bytes + 1024 > static_cast<uint32_t>(kSmemMax)) return false;
    p.div_img = FastDiv(static_cast<uint32_t>(p.Hp) * static_cast<uint32_t>(p.Wp));
    p.div_wp = FastDiv(static_cast<uint32_t>(p.Wp));
    *out = p;
    *bn_out = bn;
    return true;
}

template <int BN, int KS>
cudaError_t wide_launch_bn(const ConvArgs &a, const WidePlan &wp, const __nv_bfloat16 *W, cudaStream_t st)
{
    auto kern = halo_wide_kernel<BN, KS>;
    const CUtensorMapDataType bf = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const uint64_t K = static_cast<uint64_t>(a.KH) * a.KW * a.C;
    CUtensorMap tmap_x, tmap_w;
    // x [B][H][W][C]: one im2col load per 64-channel chunk walks the tile's
    // halo_pix positions of the padded space from the tile's first one
    const int lower[2] = {wp.lower_w, wp.lower_h};
    const int upper[2] = {wp.lower_w + a.sw * (wp.Wp - 1) - (a.W - 1), wp.lower_h + a.sh * (wp.Hp - 1) - (a.H - 1)};
    if (!halo_x_tmap(a, lower, upper, a.sw, a.sh, static_cast<int>(wp.halo_pix), &tmap_x)) return cudaErrorInvalidValue;
    {   // W [C_out][K]: boxes of 64 K x BN rows
        const uint64_t dims[2] = {K, static_cast<uint64_t>(a.C_out)};
        const uint64_t strides[1] = {K * 2};
        const uint32_t box[2] = {kBK, BN};
        if (!tc_tmap_tiled(&tmap_w, bf, 2, W, dims, strides, box)) return cudaErrorInvalidValue;
    }
    static std::mutex attr_mu;
    static bool attr_done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lk(attr_mu);
        if (!attr_done[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
            if (e != cudaSuccess) return e;
            attr_done[dev] = true;
        }
    }
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(wp.grid));
    cfg.blockDim = dim3(kWWarps * 32);
    cfg.dynamicSmemBytes = static_cast<size_t>(wp.bytes) + 1024;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a, tmap_x, tmap_w, wp);
}

template <int BN, int KS>
cudaError_t halo_launch_bn(const ConvArgs &a, const HaloPlan &hp, const __nv_bfloat16 *W, cudaStream_t st)
{
    auto kern = halo_conv_kernel<BN, KS>;
    const CUtensorMapDataType bf = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const uint64_t K = static_cast<uint64_t>(a.KH) * a.KW * a.C;
    CUtensorMap tmap_x, tmap_w, tmap_y;
    // x [B][H][W][C]: one im2col load per 64-channel chunk walks the Wp x Rh
    // halo positions of the tile (columns -pw .. W - 1 + pw of each row,
    // the padding read as zeros)
    const int lower[2] = {-a.pw, -a.ph};
    const int upper[2] = {hp.Wp - a.pw - a.W, a.Ho + (a.KH - 1) * a.dh - a.ph - a.H};
    if (!halo_x_tmap(a, lower, upper, 1, 1, hp.Wp * hp.Rh, &tmap_x)) return cudaErrorInvalidValue;
    {   // W [C_out][K]: boxes of 64 K x BN rows
        const uint64_t dims[2] = {K, static_cast<uint64_t>(a.C_out)};
        const uint64_t strides[1] = {K * 2};
        const uint32_t box[2] = {kBK, BN};
        if (!tc_tmap_tiled(&tmap_w, bf, 2, W, dims, strides, box)) return cudaErrorInvalidValue;
    }
    {   // y [B*Ho][Wo][C_out]: one output row of a 64-column atom per box
        const uint64_t dims[3] = {static_cast<uint64_t>(a.C_out), static_cast<uint64_t>(a.Wo),
                                  static_cast<uint64_t>(a.B) * a.Ho};
        const uint64_t strides[2] = {static_cast<uint64_t>(a.C_out) * 2, static_cast<uint64_t>(a.C_out) * 2 * a.Wo};
        const uint32_t box[3] = {64, static_cast<uint32_t>(a.Wo), 1};
        if (!tc_tmap_tiled(&tmap_y, bf, 3, a.y, dims, strides, box)) return cudaErrorInvalidValue;
    }
    static std::mutex attr_mu;
    static bool attr_done[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    {
        std::lock_guard<std::mutex> lk(attr_mu);
        if (!attr_done[dev]) {
            e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemMax);
            if (e != cudaSuccess) return e;
            attr_done[dev] = true;
        }
    }
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(hp.grid));
    cfg.blockDim = dim3(kWarps * 32);
    cfg.dynamicSmemBytes = static_cast<size_t>(hp.bytes) + 1024;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a, tmap_x, tmap_w, tmap_y, hp);
}

}  // namespace

// The halo form of this layer's bf16 GEMM, against the im2col GEMM's
// column tile: either form only when its column tile is at least as wide,
// since a narrower one loads every halo once per column tile where the
// im2col GEMM shares each A tile over all its columns (resident weights:
// ResNet-50's stage-2 3x3 layer at BN 64 76.8 us against BN 128 im2col
// 61 us at batch 256; streamed weights: the stride-2 stage-3 3x3 layer at
// BN 128 53.6 us against BN 256 im2col 48.7 us).  The resident form first;
// else none (the im2col GEMM).
int halo_form(const ConvArgs &a, int im2col_bn)
{
    const int sms = device_sms_or_default();
    HaloPlan hp;
    WidePlan wp;
    int bn = 0;
    if (halo_plan(a, sms, &hp, &bn) && bn >= im2col_bn) return kGemmHaloResident;
    if (wide_plan(a, sms, &wp, &bn) && bn >= im2col_bn) return kGemmHaloStreamed;
    return kGemmIm2col;
}

// The streamed form's plan geometry, for inspection: geom = {Wp, Hp, TMA
// lower corner w, h, positions per halo load, phases, taps, column tile},
// taps[kWMaxTaps] and phases[kWMaxPhases] as in WidePlan.  False when the
// layer has no streamed plan.
bool halo_streamed_geometry(const ConvArgs &a, int geom[8], uint32_t *taps, uint32_t *phases)
{
    WidePlan p;
    int bn = 0;
    if (!wide_plan(a, device_sms_or_default(), &p, &bn)) return false;
    const int g[8] = {p.Wp, p.Hp, p.lower_w, p.lower_h, static_cast<int>(p.halo_pix), p.n_ph, p.n_taps, bn};
    for (int i = 0; i < 8; ++i) geom[i] = g[i];
    for (int i = 0; i < kWMaxTaps; ++i) taps[i] = p.tap[i];
    for (int i = 0; i < kWMaxPhases; ++i) phases[i] = p.ph[i];
    return true;
}

// The halo GEMM of a bf16 layer on its decoded weights W[C_out][K] (the
// caller has checked that halo_form is not the im2col GEMM).
cudaError_t halo_gemm(const ConvArgs &a, const void *W, int im2col_bn, cudaStream_t st)
{
    int sms = 0;
    cudaError_t e = device_sm_count(&sms);
    if (e != cudaSuccess) return e;
    const __nv_bfloat16 *w = static_cast<const __nv_bfloat16 *>(W);
    // 3x3 kernels (the ResNet shapes) get the unrolled tap loop
    const bool k3 = a.KH == 3 && a.KW == 3;
    HaloPlan hp;
    int bn = 0;
    if (halo_plan(a, sms, &hp, &bn) && bn >= im2col_bn) {
        if (bn == 64) return k3 ? halo_launch_bn<64, 3>(a, hp, w, st) : halo_launch_bn<64, 0>(a, hp, w, st);
        if (bn == 128) return k3 ? halo_launch_bn<128, 3>(a, hp, w, st) : halo_launch_bn<128, 0>(a, hp, w, st);
        return k3 ? halo_launch_bn<256, 3>(a, hp, w, st) : halo_launch_bn<256, 0>(a, hp, w, st);
    }
    WidePlan wp;
    if (!wide_plan(a, sms, &wp, &bn)) return cudaErrorInvalidValue;
    const bool w3 = wp.tps == 3;           // stride-1 3x3: kernel rows as B stages, unrolled
    if (bn == 64) return w3 ? wide_launch_bn<64, 3>(a, wp, w, st) : wide_launch_bn<64, 0>(a, wp, w, st);
    return w3 ? wide_launch_bn<128, 3>(a, wp, w, st) : wide_launch_bn<128, 0>(a, wp, w, st);
}

}  // namespace onexn
