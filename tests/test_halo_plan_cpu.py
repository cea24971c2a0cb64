"""Host-side check of the streamed halo form's plan (no GPU).

The streamed form lays each image's output out in a padded space of Hp rows
of Wp positions and splits a strided layer into the phases of its input.
Each tap of Eq. 6 then reads, for the output at padded position P, the halo
load of its phase at row P - tile start + shift.  The load walks padded
positions from the tile's first one; the TMA traversal maps padded position
(r, c) to input base (lower_w + sw*c, lower_h + sh*r) and reads x at
base + the phase's offsets, zeros outside x and after the last image.

These tests take the library's own plan (onexn_conv_halo_geometry).  For
every output pixel and tap of each geometry they check that this walk
lands on exactly the input pixel the convolution reads at that tap, or on a
zero where the convolution reads padding.  They also check that the taps
cover the kernel once, that the phases partition them, that every view
stays inside one halo load, and that the traversal box is inside the TMA's
range.  The GPU parity tests check the same layers end to end."""
import numpy as np
import pytest

from paper_2105_14713_gb300 import onexn as ox

TILE = 256   # padded positions per tile

GEOMS = [
    # B, H, W, C_in, C_out, KH, KW, stride, pad, dil
    (2, 28, 28, 128, 128, 3, 3, 1, 1, 1),
    (1, 56, 56, 128, 128, 5, 5, 1, 2, 1),
    (1, 56, 56, 128, 128, 3, 3, 1, 2, 2),
    (2, 28, 28, 512, 128, 3, 1, 1, 1, 1),
    (2, 26, 28, 512, 128, 1, 3, 1, 1, 1),
    (1, 120, 120, 128, 128, 3, 3, 1, 1, 1),
    (2, 56, 56, 128, 128, 3, 3, 2, 1, 1),      # four phases of 4, 2, 2, 1 taps
    (2, 29, 29, 64, 128, 3, 3, 2, 1, 1),       # odd input size
    (1, 56, 56, 128, 128, 5, 5, 2, 2, 1),      # 25 taps in four phases
    (2, 57, 57, 128, 128, 3, 3, 2, 0, 1),      # no padding
    (1, 56, 56, 128, 128, 3, 3, 2, 2, 2),      # every tap in one phase
]


def _out(n, k, s, p, d):
    return (n + 2 * p - d * (k - 1) - 1) // s + 1


@pytest.mark.parametrize("geom", GEOMS, ids=["x".join(map(str, g[5:])) + "_%d" % g[1] for g in GEOMS])
def test_streamed_plan_reads_the_convolutions_inputs(geom):
    B, H, W, C, Co, KH, KW, s, p, d = geom
    Ho, Wo = _out(H, KH, s, p, d), _out(W, KW, s, p, d)
    g = ox.onexn_conv_halo_geometry(ox.make_desc(B, H, W, C, Co, KH, KW, s, p, d), 16, 10)
    Wp, Hp, lw, lh, halo = g["Wp"], g["Hp"], g["lower_w"], g["lower_h"], g["halo_pix"]
    assert Wp >= Wo and Hp >= Ho and g["bn"] in (64, 128)
    # the traversal box: base positions lower .. lower + s*(P - 1), corners in the TMA's range
    for lower, P, n in ((lw, Wp, W), (lh, Hp, H)):
        upper = lower + s * (P - 1) - (n - 1)
        assert -128 <= lower <= 127 and -128 <= upper <= 127
    # the taps cover the kernel once; the phases partition them in order
    assert sorted(k for k, _ in g["taps"]) == list(range(KH * KW))
    ends = [(t0, t1) for t0, t1, _, _ in g["phases"]]
    assert ends[0][0] == 0 and ends[-1][1] == KH * KW and all(a[1] == b[0] for a, b in zip(ends, ends[1:]))
    assert max(sh for _, sh in g["taps"]) + TILE <= halo <= 1024

    n_tiles = -(-B * Hp * Wp // TILE)
    P = np.arange(n_tiles * TILE)
    n, rem = np.divmod(P, Hp * Wp)
    r, c = np.divmod(rem, Wp)
    out = (n < B) & (r < Ho) & (c < Wo)              # output pixels among the positions
    checked = 0
    for t0, t1, off_w, off_h in g["phases"]:
        for ktap, shift in g["taps"][t0:t1]:
            kh, kw = divmod(ktap, KW)
            # what the plan reads: the tile's halo load of this phase, row (P - tile start) + shift
            Q = P + shift
            assert np.all((P % TILE) + shift < halo)
            qn, qrem = np.divmod(Q, Hp * Wp)
            qr, qc = np.divmod(qrem, Wp)
            xh, xw = lh + s * qr + off_h, lw + s * qc + off_w
            got_in = (qn < B) & (xh >= 0) & (xh < H) & (xw >= 0) & (xw < W)
            # what the convolution reads (Eq. 6): x[n, s*r + kh*d - p, s*c + kw*d - p]
            ih, iw = s * r + kh * d - p, s * c + kw * d - p
            want_in = (ih >= 0) & (ih < H) & (iw >= 0) & (iw < W)
            o = out
            assert np.array_equal(got_in[o], want_in[o]), (kh, kw)
            both = o & want_in
            assert np.array_equal(qn[both], n[both]) and np.array_equal(xh[both], ih[both]) and \
                np.array_equal(xw[both], iw[both]), (kh, kw)
            checked += int(o.sum())
    assert checked == B * Ho * Wo * KH * KW


@pytest.mark.parametrize("geom", [(2, 28, 28, 64, 64, 1, 1, 1, 0, 1),      # 1x1: no halo
                                  (4, 7, 7, 64, 64, 3, 3, 1, 1, 1),        # 8x8 padded for 7x7: 23% wasted
                                  (2, 14, 14, 512, 512, 3, 3, 2, 1, 1)],   # 8x8 phase space for 7x7
                         ids=["1x1", "7x7", "7x7_s2"])
def test_no_streamed_plan(geom):
    B, H, W, C, Co, KH, KW, s, p, d = geom
    with pytest.raises(ox.OnexnError) as e:
        ox.onexn_conv_halo_geometry(ox.make_desc(B, H, W, C, Co, KH, KW, s, p, d), 16, 10)
    assert e.value.status == ox.ONEXN_EUNSUPPORTED
