"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test checks one oracle function against a hand-derived value (golden
files), a closed form from the paper, brute force on tiny inputs written as
plain loops, or a special case that reduces to a library routine.  A plausible
mistake in the oracle (dropped codebook, swapped index, transposed operand,
wrong rounding, wrong tap order) fails at least one of them.
"""

import math
import os
import struct
from fractions import Fraction

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, ConvSpec, LinearSpec, make_conv, make_linear
from oracle import aq_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _h(hexstr):
    return np.frombuffer(struct.pack("<H", int(hexstr, 16)), dtype=np.float16)[0]


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append([p.strip() for p in line.split(";", 2)])
    return rows


# ----------------------------------------------------------------------------- decode
def test_decode_rule_golden_values():
    """Hand-derived fp32-sum-then-fp16 outcomes (Eq. 4 with the decode rule)."""
    for entries, expected, why in _read_golden("decode_rule_fp16.txt"):
        vals = [_h(e) for e in entries.split()]
        M = len(vals)
        cb = np.zeros((M, 256, 8), dtype=np.float16)
        for m, v in enumerate(vals):
            cb[m, 7, 3] = v                      # entry e=3 of codeword 7 in codebook m
        codes = np.full((1, 1, M), 7, dtype=np.uint8)
        W = O.decode_rule_f16(codes, cb)
        got = int(W.view(np.uint16)[0, 3])
        assert got == int(expected, 16), f"{entries}: got {got:04X}, want {expected} ({why})"
        # the other 7 entries of the group are sums of zeros
        assert np.all(W.view(np.uint16)[0, [0, 1, 2, 4, 5, 6, 7]] == 0)


def test_decode_identity_bruteforce():
    """Eq. 4: W-hat group i of row n = sum over m of codeword C^(m)[b[n,i,m]]."""
    rng = np.random.default_rng(123)
    N, G, M, g, B = 3, 4, 3, 8, 8
    cb = rng.normal(0, 0.1, size=(M, 1 << B, g)).astype(np.float16)
    codes = rng.integers(0, 1 << B, size=(N, G, M), dtype=np.uint8)
    W = O.decode_f64(codes, cb)
    assert W.shape == (N, G * g)
    for n in range(N):
        for i in range(G):
            for e in range(g):
                s = 0.0
                for m in range(M):
                    s += float(cb[m][int(codes[n][i][m])][e])
                assert W[n][i * g + e] == pytest.approx(s, rel=0, abs=1e-15)


def test_decode_codebook_order_and_element_index():
    """Exactly representable books: W[n, 8i+e] = (b0 + e)/64 - (b1 + 2e)/128."""
    cb = np.zeros((2, 256, 8), dtype=np.float16)
    for c in range(256):
        for e in range(8):
            cb[0, c, e] = (c + e) / 64.0
            cb[1, c, e] = -(c + 2 * e) / 128.0
    rng = np.random.default_rng(5)
    codes = rng.integers(0, 256, size=(5, 6, 2), dtype=np.uint8)
    Wr = O.decode_rule_f16(codes, cb).astype(np.float64)
    W64 = O.decode_f64(codes, cb)
    for n in range(5):
        for i in range(6):
            b0, b1 = int(codes[n, i, 0]), int(codes[n, i, 1])
            for e in range(8):
                want = Fraction(b0 + e, 64) - Fraction(b1 + 2 * e, 128)
                assert Fraction(W64[n, i * 8 + e]) == want
                assert Fraction(float(Wr[n, i * 8 + e])) == want


def test_decode_rule_matches_exact_sum_when_representable():
    """If the exact sum is an fp16 value, the rule returns it bit for bit."""
    cb = np.zeros((4, 256, 8), dtype=np.float16)
    for m in range(4):
        for c in range(256):
            cb[m, c, :] = np.float16((c - 128) * (1 << m))   # integers <= 1024 in magnitude
    rng = np.random.default_rng(9)
    codes = rng.integers(0, 256, size=(4, 3, 4), dtype=np.uint8)
    Wr = O.decode_rule_f16(codes, cb)
    for n in range(4):
        for i in range(3):
            s = sum((int(codes[n, i, m]) - 128) * (1 << m) for m in range(4))
            assert abs(s) <= 2048                          # exact in fp16
            assert np.all(Wr[n, i * 8:(i + 1) * 8] == np.float16(s))


def test_decode_kaq_grouping():
    """Sec. 3.1.2: one group = the 9 taps of one (cout, cin) filter."""
    rng = np.random.default_rng(3)
    Cout, Cin, M = 2, 3, 2
    cb = rng.normal(0, 0.1, size=(M, 16, 9)).astype(np.float16)
    codes = rng.integers(0, 16, size=(Cout, Cin, M), dtype=np.uint8)
    F = O.decode_kaq_f64(codes, cb)
    for o in range(Cout):
        for c in range(Cin):
            for t in range(9):
                s = float(cb[0, codes[o, c, 0], t]) + float(cb[1, codes[o, c, 1], t])
                assert F[o, c, t] == pytest.approx(s, abs=1e-15)


# ----------------------------------------------------------------------------- packing
def test_pack_layout_positions():
    """Packed byte index of code b[n, i, m]: ((kb*N + n)*8 + i%8)*M + m (8-bit codes)."""
    rng = np.random.default_rng(1)
    N, K, M = 5, 200, 3          # K/8 = 25 groups -> 4 blocks, last one has 1 group
    codes = rng.integers(0, 256, size=(N, K // 8, M), dtype=np.uint8)
    p = O.pack_codes(codes, 8)
    assert p.size == O.packed_nbytes(N, K, 8, M, 8) == 4 * N * 8 * M
    for n in range(N):
        for i in range(K // 8):
            for m in range(M):
                kb, ii = divmod(i, 8)
                assert p[((kb * N + n) * 8 + ii) * M + m] == codes[n, i, m]
    # padding groups of the last block are zero
    for n in range(N):
        for ii in range(1, 8):
            for m in range(M):
                assert p[((3 * N + n) * 8 + ii) * M + m] == 0


def test_pack_16bit_little_endian():
    codes = np.array([[[0x1234], [0xABCD]]], dtype=np.uint16)       # N=1, G=2, M=1
    p = O.pack_codes(codes, 8)
    assert p.size == O.packed_nbytes(1, 16, 8, 1, 16) == 16
    assert list(p[:4]) == [0x34, 0x12, 0xCD, 0xAB]
    assert np.all(p[4:] == 0)


# ----------------------------------------------------------------------------- activations
def test_quant_act_golden():
    for args, expected, why in _read_golden("quant_act.txt"):
        xs, ss = args.split()
        x = np.array([float(xs)], dtype=np.float16)
        got = int(O.quant_act(x, float(ss))[0])
        assert got == int(expected), f"{args}: got {got}, want {expected} ({why})"


def test_quant_act_random_bounds_and_monotone():
    x = np.sort(np.random.default_rng(0).normal(0, 3, 5000).astype(np.float16))
    q = O.quant_act(x, 0.02)
    assert q.dtype == np.int8
    assert q.min() >= -127 and q.max() <= 127
    assert np.all(np.diff(q.astype(np.int32)) >= 0)       # monotone in x
    # away from clipping, |x/s - q| <= 1/2
    inside = np.abs(x.astype(np.float64) / 0.02) < 126
    err = np.abs(x.astype(np.float64)[inside] / np.float64(np.float32(0.02)) - q[inside])
    assert err.max() <= 0.5 + 1e-5          # fp32 division can move a near-tie by 2^-24 relative


# ----------------------------------------------------------------------------- linear
def test_linear_worked_example():
    rows = {}
    with open(os.path.join(GOLDEN, "linear_worked_example.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, *v = line.split()
                rows[k] = [float(t) for t in v]
    cb = np.zeros((2, 256, 8), dtype=np.float16)
    cb[0, int(rows["code1"][0])] = rows["cb1_row3"]
    cb[1, int(rows["code2"][0])] = rows["cb2_row5"]
    codes = np.array([[[int(rows["code1"][0]), int(rows["code2"][0])]]], dtype=np.uint8)
    xq = np.array([rows["xq"]], dtype=np.int8)
    W = O.decode_f64(codes, cb)
    assert np.array_equal(W[0], np.array(rows["W"]))
    assert np.array_equal(O.decode_rule_f16(codes, cb)[0].astype(np.float64), np.array(rows["W"]))
    y = O.linear_f64(xq, rows["s_x"][0], W, np.array(rows["scale"], np.float16),
                     np.array(rows["bias"], np.float16))
    assert y.shape == (1, 1) and y[0, 0] == rows["y"][0]
    y2 = O.lut_linear_f64(xq, rows["s_x"][0], codes, cb, np.array(rows["scale"], np.float16),
                          np.array(rows["bias"], np.float16))
    assert y2[0, 0] == rows["y"][0]


def _bruteforce_linear(xq, s_x, codes, cb, scale, bias):
    """Per-codeword direct sum, never materialising W-hat (plain loops)."""
    T, K = xq.shape
    N, G, M = codes.shape
    g = cb.shape[2]
    y = np.zeros((T, N))
    for t in range(T):
        for n in range(N):
            s = 0.0
            for i in range(G):
                for m in range(M):
                    row = cb[m][int(codes[n][i][m])]
                    for e in range(g):
                        s += float(xq[t][i * g + e]) * s_x * float(row[e])
            y[t][n] = s * float(scale[n]) + (float(bias[n]) if bias is not None else 0.0)
    return y


@pytest.mark.parametrize("M,B", [(1, 8), (2, 8), (3, 8), (1, 16)])
def test_linear_bruteforce_tiny(M, B):
    inp = make_linear(LinearSpec(T=3, K=32, N=5, M=M, B=B), seed=11 + M)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y = O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"])
    yb = _bruteforce_linear(inp["xq"], inp["s_x"], inp["codes"], inp["codebooks"],
                            inp["scale"], inp["bias"])
    np.testing.assert_allclose(y, yb, rtol=1e-12, atol=1e-12)
    yl = O.lut_linear_f64(inp["xq"], inp["s_x"], inp["codes"], inp["codebooks"],
                          inp["scale"], inp["bias"])
    np.testing.assert_allclose(yl, yb, rtol=1e-12, atol=1e-12)
    # no bias
    y0 = O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], None)
    np.testing.assert_allclose(y0, yb - inp["bias"].astype(np.float64)[None, :], atol=1e-12)


def test_one_hot_codebooks_reproduce_dense_int_layer():
    """M = g = 8, C^(m)[c] = (c - 128) e_m: W-hat is any integer matrix in [-128, 127],
    i.e. a plain W8 scalar-quantized layer (Eq. 3 with z = 0).  The oracle must equal
    an int64 matmul exactly."""
    g = M = 8
    cb = np.zeros((M, 256, g), dtype=np.float16)
    for m in range(M):
        for c in range(256):
            cb[m, c, m] = c - 128
    rng = np.random.default_rng(77)
    N, K, T = 12, 64, 9
    Wint = rng.integers(-128, 128, size=(N, K))
    codes = np.zeros((N, K // g, M), dtype=np.uint8)
    for n in range(N):
        for i in range(K // g):
            for m in range(M):
                codes[n, i, m] = Wint[n, i * g + m] + 128
    W = O.decode_f64(codes, cb)
    assert np.array_equal(W, Wint.astype(np.float64))
    assert np.array_equal(O.decode_rule_f16(codes, cb).astype(np.int64), Wint)
    xq = rng.integers(-127, 128, size=(T, K)).astype(np.int8)
    ones = np.ones(N, dtype=np.float16)
    y = O.linear_f64(xq, 1.0, W, ones, None)
    assert np.array_equal(y, (xq.astype(np.int64) @ Wint.T).astype(np.float64))


def test_bits_per_weight_closed_form():
    for wl in ("tiny_linear", "qkv"):
        spec = WORKLOADS[wl]
        inp = make_linear(spec, seed=SEEDS[wl]) if wl == "tiny_linear" else None
        if inp is None:
            continue
        got = O.bits_per_weight(inp["codes"], inp["codebooks"], inp["scale"], spec.N, spec.K)
        want = O.bits_per_weight_closed_form(spec.N, spec.K, spec.g, spec.M, spec.B)
        assert got == pytest.approx(want, rel=1e-15)
    # exact rational check of the closed form on the qkv projection shape
    N, K = 2880, 960
    bits = Fraction(N * K * 2 * 8, 8) + 2 * 256 * 8 * 16 + N * 16  # codes + books + scales
    assert float(bits / (N * K)) == pytest.approx(O.bits_per_weight_closed_form(N, K, 8, 2, 8), rel=1e-15)
    assert O.bits_per_weight_closed_form(N, K, 8, 2, 8) == pytest.approx(2.04037, abs=1e-5)
    # a 2x8 layer is about 2 bits per weight (Sec. 2.4), a 1x16 layer too
    assert 2.0 < O.bits_per_weight_closed_form(4096, 4096, 8, 2, 8) < 2.01
    big = make_conv(ConvSpec(Nb=1, H=2, W=2, Cin=16, Cout=16, M=1, B=16), seed=0)
    got = O.bits_per_weight(big["codes"], big["codebooks"], big["scale"], 16, 144)
    assert got == pytest.approx(O.bits_per_weight_closed_form(16, 144, 8, 1, 16), rel=1e-15)


# ----------------------------------------------------------------------------- conv
def _bruteforce_conv(xq, s_x, W, scale, bias, kh, kw, stride, pad):
    Nb, H, Wd, Cin = xq.shape
    Cout = W.shape[0]
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (Wd + 2 * pad - kw) // stride + 1
    y = np.zeros((Nb, Ho, Wo, Cout))
    for b in range(Nb):
        for ho in range(Ho):
            for wo in range(Wo):
                for n in range(Cout):
                    s = 0.0
                    for i in range(kh):
                        for j in range(kw):
                            hi, wi = ho * stride + i - pad, wo * stride + j - pad
                            if 0 <= hi < H and 0 <= wi < Wd:
                                for c in range(Cin):
                                    s += s_x * float(xq[b, hi, wi, c]) * W[n, (i * kw + j) * Cin + c]
                    y[b, ho, wo, n] = s * float(scale[n]) + float(bias[n])
    return y


@pytest.mark.parametrize("stride", [1, 2])
def test_conv_bruteforce_tiny(stride):
    spec = ConvSpec(Nb=2, H=5, W=4, Cin=8, Cout=3, stride=stride, M=2)
    inp = make_conv(spec, seed=21 + stride)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y = O.layer_f64(inp)
    assert y.shape == (2, spec.Ho, spec.Wo, 3)
    yb = _bruteforce_conv(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"], 3, 3, stride, 1)
    np.testing.assert_allclose(y, yb, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("stride", [1, 2])
def test_conv_matches_torch_conv2d_f64(stride):
    torch = pytest.importorskip("torch")
    spec = ConvSpec(Nb=3, H=9, W=7, Cin=16, Cout=24, stride=stride, M=2)
    inp = make_conv(spec, seed=31)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y = O.layer_f64(inp)
    x = torch.from_numpy(inp["xq"].astype(np.float64) * inp["s_x"]).permute(0, 3, 1, 2)
    w = torch.from_numpy(W.reshape(24, 3, 3, 16)).permute(0, 3, 1, 2)      # OHWI -> OIHW
    ref = torch.nn.functional.conv2d(x, w, stride=stride, padding=1).permute(0, 2, 3, 1).numpy()
    ref = ref * inp["scale"].astype(np.float64) + inp["bias"].astype(np.float64)
    np.testing.assert_allclose(y, ref, rtol=1e-11, atol=1e-11)


def test_conv_centre_tap_equals_linear():
    """Only the centre tap non-zero (one-hot books) -> the conv is the linear layer on pixels."""
    Cin, Cout = 8, 4
    spec = ConvSpec(Nb=1, H=3, W=3, Cin=Cin, Cout=Cout, M=1)
    inp = make_conv(spec, seed=2)
    # rebuild codes so every non-centre tap selects an all-zero codeword (row 0)
    cb = inp["codebooks"].copy()
    cb[0, 0, :] = 0
    codes = inp["codes"].copy()
    centre = 4 * Cin // 8
    for j in range(codes.shape[1]):
        if j != centre:
            codes[:, j, 0] = 0
        else:
            codes[:, j, 0] = np.maximum(codes[:, j, 0], 1)
    W = O.decode_f64(codes, cb)
    y = O.conv2d_nhwc_f64(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"])
    Wc = W[:, 4 * Cin:5 * Cin]
    yl = O.linear_f64(inp["xq"].reshape(-1, Cin), inp["s_x"], Wc, inp["scale"], inp["bias"])
    np.testing.assert_allclose(y.reshape(-1, Cout), yl, rtol=1e-13, atol=1e-13)


def test_conv_1x1_equals_linear():
    spec = ConvSpec(Nb=2, H=3, W=5, Cin=16, Cout=8, kh=1, kw=1, pad=0, M=2)
    inp = make_conv(spec, seed=4)
    y = O.layer_f64(inp)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    yl = O.linear_f64(inp["xq"].reshape(-1, 16), inp["s_x"], W, inp["scale"], inp["bias"])
    np.testing.assert_allclose(y.reshape(-1, 8), yl, rtol=1e-13, atol=1e-13)


# ----------------------------------------------------------------------------- op counts
@pytest.mark.parametrize("M,k,Cin,Cout,h,w", [(1, 2, 2, 3, 4, 4), (2, 2, 1, 2, 3, 5)])
def test_eq_a7_op_count_and_lut_result(M, k, Cin, Cout, h, w):
    """App. A.1: the LUT kernel's counted ops equal Eq. A7, its output the dense conv."""
    rng = np.random.default_rng(M * 100 + k)
    H = rng.normal(size=(Cin, h, w))
    cb = rng.normal(size=(M, 2 ** k, 9)).astype(np.float16)
    codes = rng.integers(0, 2 ** k, size=(Cout, Cin, M), dtype=np.uint8)
    G, mults, adds = O.lut_conv_kaq_counted(H, codes, cb)
    assert (mults, adds) == O.eq_a7_flops(M, k, Cin, Cout, h, w)
    F = O.decode_kaq_f64(codes, cb).reshape(Cout, Cin, 3, 3)
    Gd, flops = O.direct_conv_counted(H, F)
    assert flops == O.eq_a2_flops(Cin, Cout, h, w)
    np.testing.assert_allclose(G, Gd, rtol=1e-12, atol=1e-12)
    # and the torch library conv agrees on the dense result
    torch = pytest.importorskip("torch")
    ref = torch.nn.functional.conv2d(torch.from_numpy(H)[None], torch.from_numpy(F), padding=1)[0]
    np.testing.assert_allclose(Gd, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_breakeven_from_eq_a7():
    """Where Eq. A7 falls below Eq. A2; the appendix's printed threshold differs."""
    for M in (1, 2, 3, 4):
        k = 8
        be = O.eq_a7_breakeven(M, k)
        c_lo, c_hi = math.floor(be), math.ceil(be)
        if c_lo == c_hi:
            c_lo -= 1
        lut = lambda co: sum(O.eq_a7_flops(M, k, 16, co, 8, 8))
        dense = lambda co: O.eq_a2_flops(16, co, 8, 8)
        assert lut(c_hi) <= dense(c_hi)
        assert lut(c_lo) > dense(c_lo)
    assert O.eq_a7_breakeven(2, 8) == 544.0
    assert O.paper_lut_breakeven(2, 8) == pytest.approx(286.875)


def _kaq_layer(Nb, H, W, Cin, Cout, M, stride, seed, n_code=16):
    """A tiny kernel-aware (g = 9) conv layer with a 16-entry codebook."""
    from aq_synth import ConvSpec
    rng = np.random.default_rng(seed)
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, stride=stride, g=9, M=M)
    return dict(codebooks=rng.normal(0, 0.1, size=(M, n_code, 9)).astype(np.float16),
                codes=rng.integers(0, n_code, size=(Cout, Cin, M), dtype=np.uint8),
                scale=rng.uniform(0.5, 1.5, size=Cout).astype(np.float16),
                bias=rng.normal(0, 0.01, size=Cout).astype(np.float16),
                xq=rng.integers(-127, 128, size=(Nb, H, W, Cin), dtype=np.int8),
                s_x=0.02, spec=spec)


def test_kaq_layer_equals_appendix_lut_kernel():
    """Sec. 3.1.2 / App. A.1: the kernel-aware conv layer (decode, OHWI layout,
    direct NHWC conv) equals the appendix's LUT kernel run image by image on the
    channels-first input, then the per-channel scale and bias."""
    inp = _kaq_layer(2, 5, 6, 3, 4, 2, 1, seed=91)
    y = O.layer_f64(inp)
    for b in range(2):
        Hc = inp["xq"][b].astype(np.float64).transpose(2, 0, 1) * inp["s_x"]
        G, _, _ = O.lut_conv_kaq_counted(Hc, inp["codes"], inp["codebooks"])
        ref = G.transpose(1, 2, 0) * inp["scale"].astype(np.float64) + inp["bias"].astype(np.float64)
        np.testing.assert_allclose(y[b], ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("stride", [1, 2])
def test_kaq_layer_equals_torch_conv_on_oihw_filters(stride):
    """kaq_ohwi is a pure relayout: the NHWC layer equals torch's NCHW conv with
    the decoded filters F [Cout][Cin][3][3] (float64)."""
    torch = pytest.importorskip("torch")
    inp = _kaq_layer(2, 7, 6, 5, 3, 3, stride, seed=92 + stride)
    y = O.layer_f64(inp)
    F = O.decode_kaq_f64(inp["codes"], inp["codebooks"]).reshape(3, 5, 3, 3)
    X = torch.from_numpy(inp["xq"].astype(np.float64).transpose(0, 3, 1, 2) * inp["s_x"])
    ref = torch.nn.functional.conv2d(X, torch.from_numpy(F), stride=stride, padding=1).numpy()
    ref = ref.transpose(0, 2, 3, 1) * inp["scale"].astype(np.float64) + inp["bias"].astype(np.float64)
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)
    # and the layout itself: W[n][t*Cin + c] = F[n][c][t]
    Wm = O.kaq_ohwi(F.reshape(3, 5, 9))
    assert Wm[2, 7 * 5 + 4] == F.reshape(3, 5, 9)[2, 4, 7]


# ----------------------------------------------------------------------------- codebook gradient
def test_input_grad_brute_force():
    """dX[t, k] = alpha * sum_n dY[t, n] * scale[n] * (sum_m C_m[b[n, k//g, m]][k % g]), with
    plain loops over every index (no matmul, no decoded matrix)."""
    rng = np.random.default_rng(71)
    T, N, Gr, g, M, n_code = 3, 5, 4, 8, 2, 16
    books = rng.normal(size=(M, n_code, g)).astype(np.float16)
    codes = rng.integers(0, n_code, size=(N, Gr, M)).astype(np.uint8)
    scale = rng.uniform(0.5, 1.5, size=N).astype(np.float16)
    dy = rng.normal(size=(T, N)).astype(np.float16)
    ref = np.zeros((T, Gr * g))
    for t in range(T):
        for k in range(Gr * g):
            acc = 0.0
            for n in range(N):
                w = 0.0
                for m in range(M):
                    w += float(books[m, codes[n, k // g, m], k % g])
                acc += float(dy[t, n]) * float(scale[n]) * w
            ref[t, k] = 0.75 * acc
    got = O.input_grad_f64(dy, codes, books, scale, alpha=0.75)
    assert np.allclose(got, ref, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("s_x", [1.0, 0.5])
def test_input_grad_is_the_derivative_of_the_layer(s_x):
    """With small-integer codebooks, scales, biases and dY (exact in float64 arithmetic), the
    loss L(xq) = sum dY * linear_f64(xq) is linear in xq, so a unit step of xq[t, k] changes L
    by exactly dL/dxq[t, k] = s_x * dL/dX[t, k] = input_grad_f64(alpha = s_x)."""
    rng = np.random.default_rng(72)
    T, N, Gr, g, M, n_code = 2, 6, 3, 8, 2, 8
    books = rng.integers(-4, 5, size=(M, n_code, g)).astype(np.float16)
    codes = rng.integers(0, n_code, size=(N, Gr, M)).astype(np.uint8)
    scale = rng.integers(1, 4, size=N).astype(np.float16)
    bias = rng.integers(-3, 4, size=N).astype(np.float16)
    dy = rng.integers(-3, 4, size=(T, N)).astype(np.float64)
    xq = rng.integers(-20, 21, size=(T, Gr * g)).astype(np.int8)
    W = O.decode_f64(codes, books)

    def loss(x):
        return float(np.sum(dy * O.linear_f64(x, s_x, W, scale, bias)))

    grad = O.input_grad_f64(dy, codes, books, scale, alpha=s_x)
    L0 = loss(xq)
    for t in range(T):
        for k in range(Gr * g):
            x1 = xq.copy()
            x1[t, k] += 1
            assert loss(x1) - L0 == grad[t, k]


def test_input_grad_of_a_unit_output_is_a_scaled_weight_row():
    """dY = e_(t, n) gives row t of dX = scale[n] * W[n, :], the other rows zero."""
    rng = np.random.default_rng(73)
    T, N, Gr, g, M = 3, 4, 2, 8, 3
    books = rng.normal(size=(M, 256, g)).astype(np.float16)
    codes = rng.integers(0, 256, size=(N, Gr, M)).astype(np.uint8)
    scale = rng.uniform(0.5, 1.5, size=N).astype(np.float16)
    W = O.decode_f64(codes, books)
    for (t, n) in ((0, 0), (2, 3), (1, 1)):
        dy = np.zeros((T, N))
        dy[t, n] = 1.0
        got = O.input_grad_f64(dy, codes, books, scale)
        want = np.zeros((T, Gr * g))
        want[t] = float(scale[n]) * W[n]
        assert np.array_equal(got, want)


def test_codebook_grad_brute_force():
    """Backward of Eq. 4: every use of codeword c in codebook m adds its group's gradient."""
    rng = np.random.default_rng(31)
    N, Gr, M, n_code, g = 3, 4, 2, 5, 8
    codes = rng.integers(0, n_code, size=(N, Gr, M), dtype=np.uint8)
    G = rng.normal(size=(N, Gr * g))
    scale = rng.uniform(0.5, 1.5, size=N).astype(np.float16)
    dC = O.codebook_grad_f64(codes, G, scale, 0.25, n_code)
    ref = np.zeros((M, n_code, g))
    for n in range(N):
        for i in range(Gr):
            for m in range(M):
                for e in range(g):
                    ref[m, codes[n, i, m], e] += 0.25 * float(scale[n]) * G[n, i * g + e]
    np.testing.assert_allclose(dC, ref, rtol=1e-14, atol=1e-14)


@pytest.mark.parametrize("kaq", [False, True])
def test_codebook_grad_is_the_derivative_of_the_decoded_layer(kaq):
    """The layer's weight term L(C) = sum_{n,k} s_x*scale[n]*G[n][k]*W-hat[n][k] is
    linear in the codebooks, so a unit step of codeword entry (m, c, e) changes L
    by exactly dC[m][c][e] (small integers keep float64 exact)."""
    rng = np.random.default_rng(32 + kaq)
    N, M, n_code = 3, 2, 4
    g, Gr = (9, 5) if kaq else (8, 3)
    books = rng.integers(-3, 4, size=(M, n_code, g)).astype(np.float64)
    codes = rng.integers(0, n_code, size=(N, Gr, M), dtype=np.uint8)
    scale = np.array([1.0, 0.5, 2.0], dtype=np.float16)
    s_x = 0.25
    if kaq:
        decode = lambda C: O.kaq_ohwi(O.decode_kaq_f64(codes, C))      # [N][9*Cin], OHWI
    else:
        decode = lambda C: O.decode_f64(codes, C)
    G = rng.integers(-4, 5, size=(N, Gr * g)).astype(np.float64)      # in decode's column order
    L = lambda C: float(np.sum(s_x * scale.astype(np.float64)[:, None] * G * decode(C)))
    Gf = O.kaq_from_ohwi(G).reshape(N, -1) if kaq else G
    dC = O.codebook_grad_f64(codes, Gf, scale, s_x, n_code)
    base = L(books)
    for m in range(M):
        for c in range(n_code):
            for e in range(g):
                C1 = books.copy()
                C1[m, c, e] += 1.0
                assert L(C1) - base == dC[m, c, e]
    assert np.array_equal(O.kaq_from_ohwi(O.kaq_ohwi(books[:, :, :9].reshape(2, 4, 9)
                                                      if kaq else np.zeros((1, 1, 9)))),
                          books[:, :, :9].reshape(2, 4, 9) if kaq else np.zeros((1, 1, 9)))


# ----------------------------------------------------------------------------- code search
def _group_err64(W, books, codes, H=None):
    """||w - w-hat||_H^2 per group in float64 (H = I when None): [N][Gr]."""
    N, Gr, M = codes.shape
    g = books.shape[2]
    E = W.astype(np.float64).reshape(N, Gr, g) - O.decode_f64(codes, books).reshape(N, Gr, g)
    if H is None:
        return np.einsum("nie,nie->ni", E, E)
    return np.einsum("nie,ief,nif->ni", E, H.astype(np.float64), E)


@pytest.mark.parametrize("weighted", [False, True])
def test_code_update_picks_the_best_codeword(weighted):
    """Each updated code is the float64 minimiser of the group error with the other
    codebooks fixed (up to float32 near-ties), and a step never raises the error."""
    rng = np.random.default_rng(41 + weighted)
    N, Gr, M, n_code, g = 4, 3, 2, 16, 8
    books = rng.normal(0, 0.5, size=(M, n_code, g)).astype(np.float16)
    W = rng.normal(0, 1, size=(N, Gr * g)).astype(np.float32)
    codes = rng.integers(0, n_code, size=(N, Gr, M), dtype=np.uint8)
    H = None
    if weighted:
        A = rng.normal(size=(Gr, g, 3 * g))
        H = np.einsum("iek,ifk->ief", A, A).astype(np.float32)      # SPD blocks of A A^T
    before = _group_err64(W, books, codes, H)
    new = O.code_update_f32(W, books, codes, H, ms=[1])
    assert np.array_equal(new[:, :, 0], codes[:, :, 0])              # only codebook 1 moves
    after = _group_err64(W, books, new, H)
    assert np.all(after <= before + 1e-9 * (1 + before))
    for n in range(N):
        for i in range(Gr):
            trial = []
            for c in range(n_code):
                cc = new.copy()
                cc[n, i, 1] = c
                trial.append(_group_err64(W, books, cc, H)[n, i])
            assert trial[new[n, i, 1]] <= min(trial) + 1e-5 * (1 + min(trial))


def test_code_update_identity_weights_equal_unweighted():
    """H = I given explicitly reproduces the unweighted step bit for bit (the
    weighted path's sums add exact zeros and unit products)."""
    rng = np.random.default_rng(43)
    N, Gr, M, n_code, g = 3, 4, 3, 32, 8
    books = rng.normal(0, 0.5, size=(M, n_code, g)).astype(np.float16)
    W = rng.normal(0, 1, size=(N, Gr * g)).astype(np.float32)
    codes = rng.integers(0, n_code, size=(N, Gr, M), dtype=np.uint8)
    I = np.broadcast_to(np.eye(g, dtype=np.float32), (Gr, g, g)).copy()
    assert np.array_equal(O.code_update_f32(W, books, codes), O.code_update_f32(W, books, codes, I))


def test_code_update_converges_to_exhaustive_on_separable_books():
    """With one codebook the step is the exhaustive search; repeated sweeps over two
    codebooks never increase the error and reach a fixed point."""
    rng = np.random.default_rng(44)
    N, Gr, n_code, g = 2, 2, 8, 8
    books1 = rng.normal(size=(1, n_code, g)).astype(np.float16)
    W = rng.normal(size=(N, Gr * g)).astype(np.float32)
    codes = np.zeros((N, Gr, 1), dtype=np.uint8)
    best = O.code_update_f32(W, books1, codes)
    for n in range(N):
        for i in range(Gr):
            errs = [np.sum((W.reshape(N, Gr, g)[n, i].astype(np.float64) - books1[0, c]) ** 2)
                    for c in range(n_code)]
            assert best[n, i, 0] == int(np.argmin(errs))
    books2 = rng.normal(size=(2, n_code, g)).astype(np.float16)
    codes = np.zeros((N, Gr, 2), dtype=np.uint8)
    err = _group_err64(W, books2, codes).sum()
    for _ in range(6):
        new = O.code_update_f32(W, books2, codes)
        e2 = _group_err64(W, books2, new).sum()
        assert e2 <= err + 1e-9
        if np.array_equal(new, codes):
            break
        codes, err = new, e2
    assert np.array_equal(O.code_update_f32(W, books2, codes), codes)
