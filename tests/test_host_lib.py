"""Host side of the C ABI (no GPU): prune / rearrange / pack / validate are
bit-exact against the oracle, argument errors are reported as status codes,
and the shared library exports every symbol include/onexn.h declares."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2105_14713_gb300 import onexn as ox
from paper_2105_14713_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "onexn.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(onexn_\w+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    names = _declared_functions()
    assert "onexn_conv_fwd" in names and "onexn_prune" in names
    lib = ctypes.CDLL(ox.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in onexn.h but not exported"
    assert set(names) == set(ox.SIGNATURES), "binding and header disagree"


def test_binding_constants_match_the_header():
    # every #define ONEXN_* and enum ONEXN_* value of include/onexn.h, evaluated
    # in C by the preprocessor's arithmetic (shifts and ors of integer literals)
    src = open(os.path.join(ROOT, "include", "onexn.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    vals = {}
    for name, expr in re.findall(r"#define[ \t]+(ONEXN_\w+)[ \t]+(.+)", src):
        expr = re.sub(r"\b(0x[0-9A-Fa-f]+|\d+)u\b", r"\1", expr.strip())
        vals[name] = eval(expr, {}, dict(vals))   # only literals and earlier ONEXN_ names
    for body in re.findall(r"typedef enum\s*\{(.*?)\}", src, flags=re.S):
        nxt = 0
        for item in body.split(","):
            item = item.strip()
            if not item:
                continue
            if "=" in item:
                n, v = (t.strip() for t in item.split("="))
                nxt = int(v, 0)
            else:
                n = item
            vals[n] = nxt
            nxt += 1
    checked = 0
    for name, v in vals.items():
        if hasattr(ox, name):
            assert getattr(ox, name) == v, name
            checked += 1
    for name in ("ONEXN_RELU", "ONEXN_ALGO_MASK", "ONEXN_ALGO_TC", "ONEXN_F32", "ONEXN_BF16", "ONEXN_ETIMEOUT",
                 "ONEXN_GRAN_KERNEL"):
        assert name in vals and hasattr(ox, name), name
    assert checked >= 15


SHAPES = [((8, 6, 3, 3), 4), ((8, 6, 3, 3), 2), ((64, 64, 1, 1), 4), ((128, 128, 3, 3), 8),
          ((32, 24, 1, 3), 16), ((12, 5, 2, 2), 3), ((16, 16, 3, 3), 16), ((24, 40, 1, 1), 1)]


@pytest.mark.parametrize("shape,N", SHAPES)
@pytest.mark.parametrize("rate", [0.0, 0.3, 0.5, 0.7, 0.9, 1.0])
@pytest.mark.parametrize("gran", [ox.ONEXN_GRAN_TAP, ox.ONEXN_GRAN_KERNEL])
def test_prune_and_pack_bitexact_vs_oracle(shape, N, rate, gran):
    rng = np.random.default_rng(hash((shape, N)) % 2**32)
    W = rng.standard_normal(shape).astype(np.float32)
    m_lib, k_lib = ox.onexn_prune(W, N, rate, gran)
    m_or, k_or = oracle.prune(W, N, rate, gran)
    assert k_lib == k_or
    np.testing.assert_array_equal(m_lib, m_or)
    for wdt, odt in ((ox.ONEXN_F32, "f32"), (ox.ONEXN_BF16, "bf16")):
        P, I, D = ox.onexn_pack(W, m_lib, N, wdt)
        Po, Io, Do = oracle.pack(W, m_or, N, odt)
        np.testing.assert_array_equal(P, Po)
        np.testing.assert_array_equal(I, Io)
        np.testing.assert_array_equal(D, Do)
        ox.onexn_packed_validate(P, I, shape[0] // N, len(I), shape[1] * shape[2] * shape[3])


def test_prune_ties_integer_weights_bitexact():
    rng = np.random.default_rng(9)
    for N in (1, 2, 4):
        W = rng.integers(-2, 3, size=(16, 12, 3, 3)).astype(np.float32)
        for rate in (0.25, 0.5, 0.75):
            for gran in (0, 1):
                a, ka = ox.onexn_prune(W, N, rate, gran)
                b, kb = oracle.prune(W, N, rate, gran)
                assert ka == kb
                np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("total", [1, 5, 9216, 147456, 4718592])
@pytest.mark.parametrize("rate", [0.0, 0.3, 0.5, 0.7, 0.9, 1.0, 0.123456789])
def test_keep_count_matches_oracle(total, rate):
    assert ox.onexn_keep_count(total, rate) == oracle.keep_count(total, rate)


@pytest.mark.parametrize("with_next", [False, True])
def test_rearrange_bitexact_vs_oracle(with_next):
    rng = np.random.default_rng(4)
    W = rng.standard_normal((48, 16, 3, 3)).astype(np.float32)
    W[5] = W[9]                        # a tie: stable order must keep 5 before 9
    Wn = rng.standard_normal((20, 48, 1, 1)).astype(np.float32) if with_next else None
    a, an, pa = ox.onexn_rearrange(W, Wn)
    b, bn, pb = oracle.rearrange(W, Wn)
    np.testing.assert_array_equal(pa, pb)
    np.testing.assert_array_equal(a, b)
    if with_next:
        np.testing.assert_array_equal(an, bn)
    assert list(pa).index(5) < list(pa).index(9)


def test_workload_config_shapes():
    c3 = wl.config3()
    assert len(c3) == 34 and c3[-1].C_out == 1280 and c3[0].H == 112
    c4 = wl.config4()
    assert len(c4) == 52 and sum(1 for l in c4 if l.KH == 3) == 16
    assert all(l.C_out % l.N == 0 for l in c3 + c4)
    assert wl.config2()[0].pixels == 64 * 28 * 28


def test_mbv2_keep_counts_closed_form():
    """kept = round((1 - rate) * C_out/N * C_in*KH*KW) on every MBv2 1x1 layer."""
    for layer in wl.config3()[:6]:
        W = wl.weights(layer.with_(B=1)).numpy()
        _, kept = ox.onexn_prune(W, layer.N, layer.rate)
        total = layer.C_out // layer.N * layer.K
        assert kept == int(np.floor((1 - layer.rate) * total + 0.5))


# ---------------------------------------------------------------- errors

def _status(fn, *a):
    with pytest.raises(ox.OnexnError) as e:
        fn(*a)
    return e.value.status


def test_prune_argument_errors():
    W = np.ones((6, 4, 1, 1), np.float32)
    assert _status(ox.onexn_prune, W, 4, 0.5) == ox.ONEXN_EINVAL         # N does not divide
    assert _status(ox.onexn_prune, W, 3, -0.1) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_prune, W, 3, 1.1) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_prune, W, 0, 0.5) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_prune, W, 3, 0.5, 7) == ox.ONEXN_EINVAL      # granularity
    assert ox.lib.onexn_prune(None, 6, 4, 1, 1, 3, 0.5, 0, None, None) == ox.ONEXN_EINVAL
    assert b"NULL" in ox.lib.onexn_last_error()


def test_pack_errors():
    W = np.ones((4, 2, 1, 1), np.float32)
    mask = np.ones((2, 2), np.uint8)
    P = np.zeros(3, np.int32)
    I = np.zeros(4, np.int32)
    D = np.zeros((4, 2), np.float32)
    t = ctypes.c_int64(0)
    p = lambda a: a.ctypes.data_as(ctypes.c_void_p)
    st = ox.lib.onexn_pack(p(W), p(mask), 4, 2, 1, 1, 2, 0, p(P), p(I), p(D), 3, ctypes.byref(t))
    assert st == ox.ONEXN_EINVAL and t.value == 4                       # t_cap too small
    mask[0, 0] = 2
    st = ox.lib.onexn_pack(p(W), p(mask), 4, 2, 1, 1, 2, 0, p(P), p(I), p(D), 4, ctypes.byref(t))
    assert st == ox.ONEXN_EINVAL
    st = ox.lib.onexn_pack(p(W), p(mask), 4, 2, 1, 1, 2, 5, p(P), p(I), p(D), 4, ctypes.byref(t))
    assert st == ox.ONEXN_EINVAL                                         # dtype


@pytest.mark.parametrize("P,I,G,t,K,frag", [
    ([1, 2], [0, 1], 1, 2, 4, "P[0]"),
    ([0, 3], [0, 1, 2], 1, 2, 4, "P[G]"),
    ([0, 2, 1], [0, 1], 2, 1, 4, "decreases"),
    ([0, 2], [1, 1], 1, 2, 4, "increasing"),
    ([0, 2], [0, 4], 1, 2, 4, "outside"),
    ([0, 1], [-1], 1, 1, 4, "outside"),
])
def test_validate_catches_corrupted_bsr(P, I, G, t, K, frag):
    with pytest.raises(ox.OnexnError) as e:
        ox.onexn_packed_validate(np.array(P), np.array(I), G, t, K)
    assert frag in str(e.value)


def test_auto_cost_model():
    # 3x3 128->128 (K = 1152, 16 groups of N = 8): the tensor-core GEMM does
    # all 128 * 1152 products per pixel after decoding the weights, the FFMA
    # kernel only the kept t * N.  On 50176 pixels the GEMM wins even at 99%
    # pruned.  On 4 pixels the FFMA kernel has 2 units of 256 pixels x 64
    # columns for 152 SMs, while the GEMM splits its 2 tiles' 36 K chunks
    # over 18 CTAs (stream-K): the GEMM wins there too.  With a tiny K
    # (8 -> 16, 3x3, one kept block) the decode launch is the larger cost.
    G, K = 128 // 8, 9 * 128
    big = ox.make_desc(64, 28, 28, 128, 128, 3, 3, 1, 1, 1)
    four = ox.make_desc(1, 2, 2, 128, 128, 3, 3, 1, 1, 1)
    for dt in (ox.ONEXN_F32, ox.ONEXN_BF16):
        ws = ox.onexn_conv_workspace_size(big, 8, G * K, dt)
        assert ox.onexn_conv_algo(big, 8, G * K // 2, dt, 0, ws) == ox.ONEXN_ALGO_TC      # 50% pruned
        assert ox.onexn_conv_algo(big, 8, G * K // 100, dt, 0, ws) == ox.ONEXN_ALGO_TC    # 99% pruned
        assert ox.onexn_conv_algo(big, 8, 0, dt, 0, ws) == ox.ONEXN_ALGO_FMA              # all pruned
        ws4 = ox.onexn_conv_workspace_size(four, 8, G * K, dt)
        assert ox.onexn_conv_algo(four, 8, G * K // 10, dt, 0, ws4) == ox.ONEXN_ALGO_TC
    tiny = ox.make_desc(1, 2, 2, 8, 16, 3, 3, 1, 1, 1)
    assert ox.onexn_conv_algo(tiny, 8, 1, ox.ONEXN_F32, 0, 1 << 20) == ox.ONEXN_ALGO_FMA
    # ... unless the caller keeps the decode for later calls
    assert ox.onexn_conv_algo(tiny, 8, 1, ox.ONEXN_F32, ox.ONEXN_REUSE_DECODE, 1 << 20) == ox.ONEXN_ALGO_TC


def test_tc_form_of_the_resnet50_stack_needs_no_gpu():
    """The GEMM form per layer of the ResNet-50 bottleneck stack (batch 256,
    bf16, 152 SMs): resident-weights halo tiles on the stage-1 3x3 layers
    (64 channels: the 3x3 x 64 x 64 weights fit in shared memory),
    streamed-weights halo tiles on the stage-2 3x3 layers (the stride-2 one
    split into its four input phases: a 29x29 padded phase space for a 28x28
    output), the im2col GEMM (128- or 256-row tiles) everywhere else: 1x1
    layers, the 256-column stage-3 layers (the halo would be loaded once per
    128-column tile) and the layers whose padding would waste over 15% of
    the positions (every 7x7 output).  The fp32 GEMM has one form."""
    forms = {}
    for l in wl.config4():
        d = ox.make_desc(l.B, l.H, l.W, l.C_in, l.C_out, l.KH, l.KW, l.stride, l.pad, l.dil)
        forms[l.name] = ox.onexn_conv_tc_form(d, 16, 10, ox.ONEXN_BF16)
        assert ox.onexn_conv_tc_form(d, 16, 10, ox.ONEXN_F32) == "im2col"
    for name, f in forms.items():
        stage, kind = name.split(".")[0], name.split("_")[-1]
        if kind == "3x3" and stage == "r50_s1":
            assert f == "halo_resident", name
        elif kind == "3x3" and stage == "r50_s2":
            assert f == "halo_streamed", name
        else:
            assert f in ("im2col", "im2col_wide"), name
    assert forms["r50_s4.b2_3x3"] == "im2col_wide" and forms["r50_s3.b2_3x3"] == "im2col"
    assert _status(ox.onexn_conv_tc_form, ox.make_desc(1, 8, 8, 6, 8, 3, 3, 1, 1, 1), 8, 10, ox.ONEXN_BF16) == \
        ox.ONEXN_EINVAL                                                      # C_in % 8 for bf16


def test_auto_batch1_mobilenet_v2_layers_pick_the_gemm():
    """Batch-1 MobileNet-V2 1x1 layers (N=4, 50%): with its workspace and the
    decode amortised (ONEXN_REUSE_DECODE, as the layer object passes), the
    tensor-core family on every layer from 28x28 down (measured on GB300:
    the FFMA kernel is 1.2-4.5x slower there, e.g. 76 vs 17 us on the 7x7
    960 -> 160 projection), in fp32 and bf16."""
    for blk in wl.config7():
        shapes = [(blk.hw, blk.c_in, blk.hidden)] if blk.hidden != blk.c_in else []
        shapes.append((blk.hw_out, blk.hidden, blk.c_out))
        for hw, ci, co in shapes:
            if hw > 28:
                continue
            d = ox.make_desc(1, hw, hw, ci, co)
            t = (co // 4) * ci // 2
            for dt in (ox.ONEXN_F32, ox.ONEXN_BF16):
                ws = ox.onexn_conv_workspace_size(d, 4, t, dt)
                assert ox.onexn_conv_algo(d, 4, t, dt, ox.ONEXN_REUSE_DECODE, ws) == ox.ONEXN_ALGO_TC, \
                    (blk.name, hw, ci, co, dt)


def test_host_entry_workspace_and_argument_checks_need_no_gpu():
    # 3x3 128->128 on 64x28x28 fp32: decoded hi/lo weights (no stream-K
    # space: chunk GEMMs may run concurrently) + 3 input and 3 output slots
    # of one chunk (64 images of 401408 bytes in ~8 MiB chunks: 3 chunks of
    # 22 images)
    d = ox.make_desc(64, 28, 28, 128, 128, 3, 3, 1, 1, 1)
    n = ox.onexn_conv_host_workspace_size(d, 8, 9216, ox.ONEXN_F32)
    img = 28 * 28 * 128 * 4
    assert n == 128 * 1152 * 8 + 3 * 2 * 22 * img
    # FFMA forced: no decoded weights
    assert ox.onexn_conv_host_workspace_size(d, 8, 9216, ox.ONEXN_F32, ox.ONEXN_ALGO_FMA) == \
        3 * 2 * 22 * img
    # bf16: half the bytes per image -> ~8 MiB chunks of 32 images
    nb = ox.onexn_conv_host_workspace_size(d, 8, 9216, ox.ONEXN_BF16)
    assert nb == 128 * 1152 * 2 + 3 * 2 * 32 * (img // 2)
    # argument errors before any device work
    st = ox.lib.onexn_conv_fwd_host(ctypes.byref(d), None, None, None, 8, 9216, None, None, None,
                                    ox.ONEXN_F32, 0, None, 0, None)
    assert st == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_host_workspace_size, d, 3, 10, ox.ONEXN_F32) == ox.ONEXN_EINVAL


def test_conv_shape_and_argument_errors_need_no_gpu():
    d = ox.make_desc(2, 7, 7, 8, 16, 3, 3, 2, 1, 1)
    assert ox.onexn_conv_out_shape(d) == (4, 4)
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_F32) == ox.ONEXN_ALGO_FMA
    # tcgen05 family: the decoded weights (bf16: 2 bytes per weight; fp32:
    # hi and lo tf32 parts, 8 bytes), plus the stream-K space (one
    # 128 x BN fp32 partial slot per CTA for 152 CTAs, and 152 flags) that
    # the reported size includes; the weights alone are the minimum.
    sk = 152 * 128 * 64 * 4 + 768
    w16, w32 = 16 * 9 * 8 * 2, 16 * 9 * 8 * 8
    assert w16 % 256 == 0 and w32 % 256 == 0
    assert ox.onexn_conv_workspace_size(d, 8, 100, ox.ONEXN_BF16) == w16 + sk
    assert ox.onexn_conv_workspace_size(d, 8, 100, ox.ONEXN_F32) == w32 + sk
    # bf16: the tcgen05 family when the weights fit, else FFMA
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_BF16, 0, w16) == ox.ONEXN_ALGO_TC
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_BF16, 0, w16 - 1) == ox.ONEXN_ALGO_FMA
    assert ox.onexn_conv_workspace_size(d, 8, 100, ox.ONEXN_F32, ox.ONEXN_ALGO_FMA) == 0
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_F32, 0, w32 - 1) == ox.ONEXN_ALGO_FMA
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_F32, ox.ONEXN_ALGO_TC, w32) == ox.ONEXN_ALGO_TC
    assert _status(ox.onexn_conv_algo, d, 8, 100, ox.ONEXN_BF16, ox.ONEXN_ALGO_TC, 0) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_algo, d, 8, 100, ox.ONEXN_F32, ox.ONEXN_ALGO_TC, w32 - 1) == \
        ox.ONEXN_EINVAL
    # C_out not a multiple of 8: no tensor-core tiles; AUTO falls back to FFMA
    d12 = ox.make_desc(1, 4, 4, 8, 12)
    for dt in (ox.ONEXN_F32, ox.ONEXN_BF16):
        assert _status(ox.onexn_conv_algo, d12, 4, 1, dt, ox.ONEXN_ALGO_TC, 1 << 30) == ox.ONEXN_EUNSUPPORTED
        assert ox.onexn_conv_algo(d12, 4, 1, dt, 0, 1 << 30) == ox.ONEXN_ALGO_FMA
        assert ox.onexn_conv_workspace_size(d12, 4, 1, dt) == 0
    bad = ox.make_desc(1, 2, 2, 8, 16, 5, 5)
    assert _status(ox.onexn_conv_out_shape, bad) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_algo, d, 3, 10, ox.ONEXN_F32) == ox.ONEXN_EINVAL    # N | C_out
    d6 = ox.make_desc(1, 4, 4, 6, 16)
    assert _status(ox.onexn_conv_algo, d6, 8, 10, ox.ONEXN_F32) == ox.ONEXN_EINVAL   # C_in % 4
    assert _status(ox.onexn_conv_algo, d, 8, 10**9, ox.ONEXN_F32) == ox.ONEXN_EINVAL  # t > G*K
    assert _status(ox.onexn_conv_algo, d, 8, 10, 7) == ox.ONEXN_EINVAL               # dtype
    assert _status(ox.onexn_conv_algo, d, 8, 10, 0, 1 << 20) == ox.ONEXN_EINVAL      # flags
    # conv_fwd rejects bad pointers before touching the GPU
    st = ox.lib.onexn_conv_fwd(ctypes.byref(d), None, None, None, 8, 0, None, None, None, 0, 0,
                               None, 0, None)
    assert st == ox.ONEXN_EINVAL
    buf = (ctypes.c_char * 64)()
    base = ctypes.addressof(buf)
    mis = ctypes.c_void_p(base + (16 - base % 16) % 16 + 4)
    st = ox.lib.onexn_conv_fwd(ctypes.byref(d), mis, mis, mis, 8, 1, mis, mis, None, 0, 0, None, 0,
                               None)
    assert st == ox.ONEXN_EINVAL and b"aligned" in ox.lib.onexn_last_error()


def _aligned_host(nbytes, align=256):
    buf = (ctypes.c_char * (nbytes + align))()
    base = ctypes.addressof(buf)
    return buf, base + (align - base % align) % align


def test_conv_fwd_ex_residual_errors_need_no_gpu():
    """The residual operand must be 16-byte aligned and either be y or not
    overlap it; both are refused before the GPU is touched."""
    d = ox.make_desc(1, 4, 4, 8, 16)                   # 16 pixels x 16 channels
    keep, base = _aligned_host(1 << 16)
    P, I, D = base, base + 256, base + 512
    x, y = base + 1024, base + 8192                     # y: 16*16*4 = 1 KiB
    ex = ox.lib.onexn_conv_fwd_ex
    for r, what in ((y + 4, b"aligned"), (y + 16, b"overlaps"), (y - 512, b"overlaps")):
        st = ex(ctypes.byref(d), P, I, D, 8, 1, x, y, None, r, ox.ONEXN_F32, 0, None, 0, None)
        assert st == ox.ONEXN_EINVAL and what in ox.lib.onexn_last_error(), ox.lib.onexn_last_error()
    st = ex(ctypes.byref(d), P, I, D, 8, 1, x, y, None, y, ox.ONEXN_F32, 1 << 20, None, 0, None)
    assert st == ox.ONEXN_EINVAL                         # unknown flag bit


def test_dwconv_argument_errors_need_no_gpu():
    keep, base = _aligned_host(1 << 16)
    W, x, y = base, base + 4096, base + 32768
    dw = ox.lib.onexn_dwconv_fwd
    cases = [
        (ox.make_desc(1, 4, 4, 16, 32, 3, 3, 1, 1, 1), ox.ONEXN_F32, 0, x, y, b"differ"),
        (ox.make_desc(1, 4, 4, 6, 6, 3, 3, 1, 1, 1), ox.ONEXN_F32, 0, x, y, b"multiple"),
        (ox.make_desc(1, 4, 4, 12, 12, 3, 3, 1, 1, 1), ox.ONEXN_BF16, 0, x, y, b"multiple"),
        (ox.make_desc(1, 4, 4, 16, 16, 3, 3, 1, 1, 1), ox.ONEXN_F32, 1 << 20, x, y, b"flags"),
        (ox.make_desc(1, 4, 4, 16, 16, 3, 3, 1, 1, 1), ox.ONEXN_F32, 0, x, x + 512, b"overlap"),
        (ox.make_desc(1, 4, 4, 16, 16, 3, 3, 1, 1, 1), ox.ONEXN_F32, 0, x + 8, y, b"aligned"),
        (ox.make_desc(1, 4, 4, 16, 16, 3, 3, 1, 1, 1), 5, 0, x, y, b"dtype"),
    ]
    for d, dt, fl, xp, yp, what in cases:
        st = dw(ctypes.byref(d), W, None, xp, yp, dt, fl, None)
        assert st == ox.ONEXN_EINVAL and what in ox.lib.onexn_last_error(), ox.lib.onexn_last_error()
    # an empty batch is a no-op that needs no device
    d0 = ox.make_desc(0, 4, 4, 16, 16, 3, 3, 1, 1, 1)
    assert dw(ctypes.byref(d0), None, None, None, None, ox.ONEXN_F32, 0, None) == ox.ONEXN_OK


def test_decoded_flag_selects_tc_and_is_checked():
    """ONEXN_DECODED (weights already decoded in the workspace) implies the
    tc family: AUTO resolves to it, another forced family is EINVAL, the
    workspace must still hold the decoded weights, and the host-memory and
    allocation-free entries refuse it."""
    d = ox.make_desc(2, 7, 7, 8, 16, 3, 3, 1, 1, 1)
    w32 = 16 * 9 * 8 * 8
    D = ox.ONEXN_DECODED
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_F32, D, w32) == ox.ONEXN_ALGO_TC
    assert ox.onexn_conv_algo(d, 8, 100, ox.ONEXN_F32, D | ox.ONEXN_ALGO_TC, w32) == ox.ONEXN_ALGO_TC
    tiny = ox.make_desc(1, 2, 2, 8, 16, 3, 3, 1, 1, 1)           # AUTO alone would pick FFMA here
    assert ox.onexn_conv_algo(tiny, 8, 1, ox.ONEXN_F32, 0, w32) == ox.ONEXN_ALGO_FMA
    assert ox.onexn_conv_algo(tiny, 8, 1, ox.ONEXN_F32, D, w32) == ox.ONEXN_ALGO_TC
    assert _status(ox.onexn_conv_algo, d, 8, 100, ox.ONEXN_F32, D | ox.ONEXN_ALGO_FMA, w32) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_algo, d, 8, 100, ox.ONEXN_F32, D, w32 - 1) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_host_workspace_size, d, 8, 100, ox.ONEXN_F32, D) == ox.ONEXN_EINVAL
    assert _status(ox.onexn_conv_host_workspace_size, d, 8, 100, ox.ONEXN_F32, ox.ONEXN_REUSE_DECODE) == \
        ox.ONEXN_EINVAL
    st = ox.lib.onexn_conv_fwd_noalloc(ctypes.byref(d), None, None, None, 8, 100, None, None, None,
                                       ox.ONEXN_F32, D, None)
    assert st == ox.ONEXN_EINVAL and b"DECODED" in ox.lib.onexn_last_error()


def test_device_prune_and_pack_argument_errors_need_no_gpu():
    n = ctypes.c_size_t(0)
    assert ox.lib.onexn_prune_device_workspace_size(64, 32, 3, 3, 8, ox.ONEXN_GRAN_TAP, ctypes.byref(n)) == 0
    assert n.value >= 8 * 9 * 32 * 8 and n.value % 256 == 0
    assert ox.lib.onexn_prune_device_workspace_size(64, 32, 3, 3, 7, 0, ctypes.byref(n)) == ox.ONEXN_EINVAL
    assert ox.lib.onexn_prune_device_workspace_size(64, 32, 3, 3, 8, 5, ctypes.byref(n)) == ox.ONEXN_EINVAL
    keep, base = _aligned_host(1 << 20)
    kept = ctypes.c_int64(0)
    f = ox.lib.onexn_prune_device
    assert f(base, 64, 32, 3, 3, 8, 1.5, 0, base, ctypes.byref(kept), base, 1 << 20, None) == ox.ONEXN_EINVAL
    assert f(base, 64, 32, 3, 3, 8, 0.5, 0, base, ctypes.byref(kept), base, 16, None) == ox.ONEXN_EINVAL
    assert b"workspace" in ox.lib.onexn_last_error()
    assert f(base, 64, 32, 3, 3, 8, 0.5, 0, None, ctypes.byref(kept), base, 1 << 20, None) == ox.ONEXN_EINVAL
    assert f(base, 64, 32, 3, 3, 8, 0.5, 0, base, ctypes.byref(kept), base + 8, 1 << 19, None) == \
        ox.ONEXN_EINVAL
    assert ox.lib.onexn_pack_device_workspace_size(64, 8, ctypes.byref(n)) == 0 and n.value == 256
    g = ox.lib.onexn_pack_device
    assert g(base, base, 64, 32, 3, 3, 8, 7, base, base, base, 10, base, 256, None) == ox.ONEXN_EINVAL
    assert g(base, base, 64, 32, 3, 3, 8, 0, base, None, None, 10, base, 256, None) == ox.ONEXN_EINVAL
    assert g(base, base, 64, 32, 3, 3, 8, 0, base, base, base, 10, base, 4, None) == ox.ONEXN_EINVAL


def test_bwd_workspace_sizes_show_the_input_gradient_path():
    """Input gradient: decoded weights + their flipped transpose; a strided
    layer runs on the tensor cores over dy dilated by the stride (its
    buffer is in the workspace), padding beyond d(K-1) on the direct kernel
    (no extra buffer).  Weight gradient: transposed im2col, transposed dy
    (fp32: tf32 hi and lo), column sums, GEMM partial tiles."""
    wb = lambda co, k, es: -(-co * k * es // 256) * 256
    r256 = lambda v: -(-v // 256) * 256
    d1 = ox.make_desc(2, 15, 13, 32, 64, 3, 3, 1, 1, 1)
    assert ox.onexn_conv_bwd_data_workspace_size(d1, 8, 100, ox.ONEXN_F32) == 2 * wb(64, 288, 8)
    d2 = ox.make_desc(3, 15, 13, 32, 64, 3, 3, 2, 1, 1)            # Ho, Wo = 8, 7: dilated 15 x 13
    assert ox.onexn_conv_bwd_data_workspace_size(d2, 8, 100, ox.ONEXN_F32) == \
        2 * wb(64, 288, 8) + r256(3 * 15 * 13 * 64 * 4)
    assert ox.onexn_conv_bwd_data_workspace_size(d2, 8, 100, ox.ONEXN_BF16) == \
        2 * wb(64, 288, 2) + r256(3 * 15 * 13 * 64 * 2)
    d3 = ox.make_desc(2, 14, 14, 64, 128, 1, 1, 2, 0, 1)           # 1x1 s2: 7 x 7 -> dilated 13 x 13 + 1
    assert ox.onexn_conv_bwd_data_workspace_size(d3, 4, 100, ox.ONEXN_F32) == \
        2 * wb(128, 64, 8) + r256(2 * 14 * 14 * 128 * 4)
    d4 = ox.make_desc(2, 13, 11, 32, 64, 3, 3, 2, 3, 1)            # pad 3 > d(K-1): direct kernel
    assert ox.onexn_conv_bwd_data_workspace_size(d4, 8, 100, ox.ONEXN_F32) == 2 * wb(64, 288, 8)
    # weight gradient on 2 x 15 x 13 -> P = 390 pixels, padded to 448
    n = ox.onexn_conv_bwd_weight_workspace_size(d1, 8, ox.ONEXN_F32)
    K, Pp = 288, 448
    base = r256(K * Pp * 4) + 2 * r256(64 * Pp * 4) + r256(64 * (Pp // 32) * 4)
    assert n > base and (n - base) % (128 * 64 * 4) == 0           # whole 128 x 64 fp32 partial tiles
    with pytest.raises(ox.OnexnError):
        ox.onexn_conv_bwd_data_workspace_size(ox.make_desc(1, 4, 4, 8, 12), 4, 1, ox.ONEXN_F32)   # C_out % 8


def test_dwproj_argument_errors_need_no_gpu():
    keep, base = _aligned_host(1 << 16)
    f = ox.lib.onexn_dwproj_fwd
    def call(desc, dtype=ox.ONEXN_F32, flags=0, C_out=32, W=base):
        return f(ctypes.byref(desc), W, None, base, base, base, 4, 10, C_out, base, base + 32768, None, None,
                 dtype, flags, None, 0, None)
    assert call(ox.make_desc(1, 8, 8, 64, 64, 3, 3, 3, 1, 1)) == ox.ONEXN_EINVAL           # stride 3
    assert call(ox.make_desc(1, 8, 8, 64, 64, 5, 5, 1, 2, 1)) == ox.ONEXN_EINVAL           # 5x5
    assert call(ox.make_desc(1, 8, 8, 64, 32, 3, 3, 1, 1, 1)) == ox.ONEXN_EINVAL           # C_in != C_out
    assert call(ox.make_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 1), dtype=ox.ONEXN_BF16) == ox.ONEXN_EUNSUPPORTED
    assert call(ox.make_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 1), flags=ox.ONEXN_ALGO_FMA) == ox.ONEXN_EINVAL
    st = call(ox.make_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 1), W=base + 4)                    # misaligned W_dw
    assert st == ox.ONEXN_EINVAL and b"aligned" in ox.lib.onexn_last_error()
    st = call(ox.make_desc(1, 8, 8, 64, 64, 3, 3, 1, 1, 1))                                # no workspace
    assert st == ox.ONEXN_EINVAL and b"workspace" in ox.lib.onexn_last_error()
