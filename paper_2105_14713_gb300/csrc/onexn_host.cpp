// Host side of the onexn C ABI: the offline steps of 1xN pruning that run
// once per layer before inference -- block scoring and selection (Sec. 3.2,
// Eq. 4-5), filter rearrangement (Sec. 3.3) and BSR encoding (Sec. 3.4) --
// plus argument checking and the thread-local error message.
//
// These are O(C_out * C_in * KH * KW) integer and sort work; they produce the
// (P, I, D) arrays that the caller copies to the device once.
#include "onexn.h"
#include "onexn_internal.h"

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <numeric>
#include <vector>

namespace onexn {

static thread_local char g_err[512];

onexn_status fail(onexn_status st, const char *fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return st;
}

void clear_error() { g_err[0] = 0; }

const char *last_error() { return g_err; }

// Round-to-nearest-even fp32 -> bfloat16 bits (finite inputs).
uint16_t bf16_bits_rne(float f)
{
    uint32_t u;
    std::memcpy(&u, &f, sizeof(u));
    const uint32_t round = 0x7fffu + ((u >> 16) & 1u);
    return static_cast<uint16_t>((u + round) >> 16);
}

}  // namespace onexn

using onexn::fail;

extern "C" const char *onexn_last_error(void) { return onexn::last_error(); }

extern "C" int onexn_version(void) { return (1 << 16) | 0; }

extern "C" onexn_status onexn_keep_count(int64_t total_blocks, double rate, int64_t *keep)
{
    onexn::clear_error();
    if (!keep) return fail(ONEXN_EINVAL, "keep_count: keep is NULL");
    if (total_blocks < 0) return fail(ONEXN_EINVAL, "keep_count: total_blocks < 0");
    if (!(rate >= 0.0 && rate <= 1.0))
        return fail(ONEXN_EINVAL, "keep_count: rate %g outside [0, 1]", rate);
    // Rate at 1e-6 resolution; keep = floor(total * kept_ppm / 1e6 + 1/2).
    const int64_t kept_ppm = 1000000 - static_cast<int64_t>(std::llround(rate * 1e6));
    if (total_blocks > (INT64_MAX - 500000) / 1000000)
        return fail(ONEXN_EINVAL, "keep_count: total_blocks too large");
    *keep = (total_blocks * kept_ppm + 500000) / 1000000;
    return ONEXN_OK;
}

static bool dims_ok(int C_out, int C_in, int KH, int KW)
{
    return C_out > 0 && C_in > 0 && KH > 0 && KW > 0 &&
           static_cast<int64_t>(KH) * KW * C_in < (int64_t(1) << 30) &&
           static_cast<int64_t>(C_out) * C_in * KH * KW < (int64_t(1) << 40);
}

extern "C" onexn_status onexn_prune(const float *W, int C_out, int C_in, int KH, int KW, int N,
                                    double rate, int gran, uint8_t *mask, int64_t *kept)
{
    onexn::clear_error();
    if (!W || !mask || !kept) return fail(ONEXN_EINVAL, "prune: NULL pointer");
    if (!dims_ok(C_out, C_in, KH, KW)) return fail(ONEXN_EINVAL, "prune: bad dimensions");
    if (N < 1 || C_out % N) return fail(ONEXN_EINVAL, "prune: N=%d must divide C_out=%d", N, C_out);
    if (gran != ONEXN_GRAN_TAP && gran != ONEXN_GRAN_KERNEL)
        return fail(ONEXN_EINVAL, "prune: unknown granularity %d", gran);
    const int G = C_out / N;
    const int T = KH * KW;                 // taps
    const int K = T * C_in;                // index space
    const int nb = gran == ONEXN_GRAN_TAP ? K : C_in;
    const int64_t total = static_cast<int64_t>(G) * nb;
    int64_t keep = 0;
    onexn_status st = onexn_keep_count(total, rate, &keep);
    if (st != ONEXN_OK) return st;

    std::vector<double> score;
    std::vector<int64_t> order;
    try {
        score.resize(total);
        order.resize(total);
    } catch (const std::bad_alloc &) {
        return fail(ONEXN_ENOMEM, "prune: cannot allocate %lld scores", (long long)total);
    }
    // Scores, block-major.  Same per-block summation order in both modes:
    // n outer, then (kh, kw) for the kernel granularity.
    const int64_t ostride = static_cast<int64_t>(C_in) * T;   // one filter
    for (int g = 0; g < G; ++g) {
        double *sg = score.data() + static_cast<int64_t>(g) * nb;
        if (gran == ONEXN_GRAN_TAP) {
            for (int k = 0; k < K; ++k) sg[k] = 0.0;
            for (int n = 0; n < N; ++n) {
                const float *wo = W + (static_cast<int64_t>(g) * N + n) * ostride;
                for (int c = 0; c < C_in; ++c)
                    for (int t = 0; t < T; ++t)
                        sg[t * C_in + c] += std::fabs(static_cast<double>(wo[c * T + t]));
            }
        } else {
            for (int c = 0; c < C_in; ++c) sg[c] = 0.0;
            for (int n = 0; n < N; ++n) {
                const float *wo = W + (static_cast<int64_t>(g) * N + n) * ostride;
                for (int c = 0; c < C_in; ++c) {
                    double s = sg[c];
                    for (int t = 0; t < T; ++t) s += std::fabs(static_cast<double>(wo[c * T + t]));
                    sg[c] = s;
                }
            }
        }
    }
    // Select the `keep` best blocks: larger score first, lower index on ties.
    std::iota(order.begin(), order.end(), int64_t(0));
    auto better = [&](int64_t a, int64_t b) {
        return score[a] > score[b] || (score[a] == score[b] && a < b);
    };
    if (keep > 0 && keep < total)
        std::nth_element(order.begin(), order.begin() + (keep - 1), order.end(), better);
    std::memset(mask, 0, static_cast<size_t>(G) * K);
    if (keep > 0) {
        // Everything at or before position keep-1 (after nth_element) is kept.
        for (int64_t i = 0; i < keep; ++i) {
            const int64_t blk = order[i];
            const int64_t g = blk / nb, b = blk % nb;
            if (gran == ONEXN_GRAN_TAP) {
                mask[g * K + b] = 1;
            } else {
                for (int t = 0; t < T; ++t) mask[g * K + static_cast<int64_t>(t) * C_in + b] = 1;
            }
        }
    }
    *kept = keep;
    return ONEXN_OK;
}

extern "C" onexn_status onexn_rearrange(float *W_l, int C_out, int C_in, int KH, int KW,
                                        float *W_next, int C_out_next, int KH_next,
                                        int KW_next, int32_t *perm)
{
    onexn::clear_error();
    if (!W_l || !perm) return fail(ONEXN_EINVAL, "rearrange: NULL pointer");
    if (!dims_ok(C_out, C_in, KH, KW)) return fail(ONEXN_EINVAL, "rearrange: bad dimensions");
    if (W_next && !dims_ok(C_out_next, C_out, KH_next, KW_next))
        return fail(ONEXN_EINVAL, "rearrange: bad next-layer dimensions");
    const int64_t fs = static_cast<int64_t>(C_in) * KH * KW;
    std::vector<double> l1;
    std::vector<int32_t> idx;
    std::vector<float> tmp;
    try {
        l1.assign(C_out, 0.0);
        idx.resize(C_out);
        tmp.resize(static_cast<size_t>(C_out) * fs);
    } catch (const std::bad_alloc &) {
        return fail(ONEXN_ENOMEM, "rearrange: allocation failed");
    }
    for (int o = 0; o < C_out; ++o) {
        const float *w = W_l + o * fs;
        double s = 0.0;
        for (int64_t e = 0; e < fs; ++e) s += std::fabs(static_cast<double>(w[e]));
        l1[o] = s;
    }
    std::iota(idx.begin(), idx.end(), 0);
    std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) { return l1[a] > l1[b]; });
    std::memcpy(perm, idx.data(), sizeof(int32_t) * C_out);

    std::memcpy(tmp.data(), W_l, sizeof(float) * tmp.size());
    for (int o = 0; o < C_out; ++o)
        std::memcpy(W_l + o * fs, tmp.data() + perm[o] * fs, sizeof(float) * fs);

    if (W_next) {
        const int64_t ks = static_cast<int64_t>(KH_next) * KW_next;
        std::vector<float> row(static_cast<size_t>(C_out) * ks);
        for (int j = 0; j < C_out_next; ++j) {
            float *wj = W_next + j * C_out * ks;
            std::memcpy(row.data(), wj, sizeof(float) * row.size());
            for (int o = 0; o < C_out; ++o)
                std::memcpy(wj + o * ks, row.data() + perm[o] * ks, sizeof(float) * ks);
        }
    }
    return ONEXN_OK;
}

extern "C" onexn_status onexn_pack(const float *W, const uint8_t *mask, int C_out, int C_in,
                                   int KH, int KW, int N, int wdtype, int32_t *P, int32_t *I,
                                   void *D, int64_t t_cap, int64_t *t)
{
    onexn::clear_error();
    if (!W || !mask || !P || !t || (t_cap > 0 && (!I || !D)))
        return fail(ONEXN_EINVAL, "pack: NULL pointer");
    if (!dims_ok(C_out, C_in, KH, KW)) return fail(ONEXN_EINVAL, "pack: bad dimensions");
    if (N < 1 || C_out % N) return fail(ONEXN_EINVAL, "pack: N=%d must divide C_out=%d", N, C_out);
    if (wdtype != ONEXN_F32 && wdtype != ONEXN_BF16)
        return fail(ONEXN_EINVAL, "pack: unknown weight dtype %d", wdtype);
    const int G = C_out / N, T = KH * KW, K = T * C_in;
    // Count first so that a short buffer is reported before anything is written.
    int64_t cnt = 0;
    for (int64_t e = 0; e < static_cast<int64_t>(G) * K; ++e) {
        if (mask[e] > 1) return fail(ONEXN_EINVAL, "pack: mask byte %lld is %d", (long long)e, mask[e]);
        cnt += mask[e];
    }
    *t = cnt;
    if (cnt > t_cap)
        return fail(ONEXN_EINVAL, "pack: t_cap=%lld < kept blocks %lld", (long long)t_cap,
                    (long long)cnt);
    if (cnt > INT32_MAX) return fail(ONEXN_EINVAL, "pack: too many blocks for int32 P");
    float *Df = static_cast<float *>(D);
    uint16_t *Dh = static_cast<uint16_t *>(D);
    const int64_t ostride = static_cast<int64_t>(C_in) * T;
    int64_t z = 0;
    for (int g = 0; g < G; ++g) {
        P[g] = static_cast<int32_t>(z);
        const uint8_t *mg = mask + static_cast<int64_t>(g) * K;
        for (int k = 0; k < K; ++k) {
            if (!mg[k]) continue;
            const int tap = k / C_in, c = k - tap * C_in;
            I[z] = k;
            const float *src = W + static_cast<int64_t>(g) * N * ostride + c * T + tap;
            if (wdtype == ONEXN_F32) {
                for (int n = 0; n < N; ++n) Df[z * N + n] = src[n * ostride];
            } else {
                for (int n = 0; n < N; ++n) Dh[z * N + n] = onexn::bf16_bits_rne(src[n * ostride]);
            }
            ++z;
        }
    }
    P[G] = static_cast<int32_t>(z);
    return ONEXN_OK;
}

extern "C" onexn_status onexn_packed_validate(const int32_t *P, const int32_t *I, int G, int64_t t,
                                              int K)
{
    onexn::clear_error();
    if (!P || (t > 0 && !I)) return fail(ONEXN_EINVAL, "validate: NULL pointer");
    if (G < 1 || K < 1 || t < 0) return fail(ONEXN_EINVAL, "validate: bad sizes");
    if (P[0] != 0) return fail(ONEXN_EINVAL, "validate: P[0]=%d, expected 0", P[0]);
    if (P[G] != t) return fail(ONEXN_EINVAL, "validate: P[G]=%d, expected t=%lld", P[G], (long long)t);
    for (int g = 0; g < G; ++g) {
        if (P[g + 1] < P[g])
            return fail(ONEXN_EINVAL, "validate: P decreases at group %d", g);
        int32_t prev = -1;
        for (int32_t z = P[g]; z < P[g + 1]; ++z) {
            if (I[z] < 0 || I[z] >= K)
                return fail(ONEXN_EINVAL, "validate: I[%d]=%d outside [0, %d)", z, I[z], K);
            if (I[z] <= prev)
                return fail(ONEXN_EINVAL, "validate: I not increasing in group %d at %d", g, z);
            prev = I[z];
        }
    }
    return ONEXN_OK;
}

extern "C" onexn_status onexn_conv_out_shape(const onexn_conv_desc *d, int *Ho, int *Wo)
{
    onexn::clear_error();
    if (!d || !Ho || !Wo) return fail(ONEXN_EINVAL, "out_shape: NULL pointer");
    if (d->B < 0 || d->H < 1 || d->W < 1 || d->C_in < 1 || d->C_out < 1 || d->KH < 1 ||
        d->KW < 1 || d->stride_h < 1 || d->stride_w < 1 || d->pad_h < 0 || d->pad_w < 0 ||
        d->dil_h < 1 || d->dil_w < 1)
        return fail(ONEXN_EINVAL, "conv: invalid geometry");
    const int64_t eh = static_cast<int64_t>(d->H) + 2 * d->pad_h - static_cast<int64_t>(d->dil_h) * (d->KH - 1) - 1;
    const int64_t ew = static_cast<int64_t>(d->W) + 2 * d->pad_w - static_cast<int64_t>(d->dil_w) * (d->KW - 1) - 1;
    if (eh < 0 || ew < 0) return fail(ONEXN_EINVAL, "conv: kernel larger than padded input");
    *Ho = static_cast<int>(eh / d->stride_h + 1);
    *Wo = static_cast<int>(ew / d->stride_w + 1);
    return ONEXN_OK;
}
