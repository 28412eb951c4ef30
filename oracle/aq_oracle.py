"""CPU oracle for the additive-quantized (AQ) weight x 8-bit activation layer.

TEST INFRASTRUCTURE ONLY.  Nothing in the product library imports, links or
executes this file: only the tests, the smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the CUDA path; the two meet only
through the seeded arrays of ``aq_synth``.

Everything here is the plain definition, in float64 unless a function states a
narrower precision on purpose (the bit-exact decode rule and the activation
quantizer, whose integer/fp16 outcomes must be decided in the same precision as
the GPU).  numpy fancy indexing (gather) and matmul are the only library
primitives used.

Notation (paper Sec. 2.4, Eq. 4 and App. A.1 Eq. A3):
  g        group size (weights per group)
  M        number of codebooks C^(1..M), each with 2**B rows of g entries
  b[i, m]  integer code of group i in codebook m, in [0, 2**B)
  W-hat    concatenation over groups i of  sum_m C^(m)[b[i, m]]
Groups enumerate the weight matrix row-major: row n, then k // g.

Function pinning: every function is pinned by tests/test_oracle_pins.py
(closed forms, hand-derived values in tests/golden/, brute force on tiny
inputs, library special cases).  No function is parity-unpinned.
"""

from __future__ import annotations

import math

import numpy as np

__all__ = [
    "decode_f64", "decode_rule_f16", "decode_kaq_f64", "kaq_ohwi", "kaq_from_ohwi",
    "codebook_grad_f64", "input_grad_f64", "code_update_f32", "pack_codes", "packed_nbytes",
    "quant_act", "linear_f64", "conv2d_nhwc_f64", "lut_linear_f64",
    "lut_conv_kaq_counted", "direct_conv_counted", "eq_a7_flops", "eq_a2_flops",
    "paper_lut_breakeven", "eq_a7_breakeven", "bits_per_weight",
    "bits_per_weight_closed_form", "layer_f64", "compare",
]

# Codes per packed block along K (one 64-wide K block of the GPU tiles holds
# 64 // g groups).  The packed layout is the GPU library's storage format; the
# oracle writes it out from its definition so that the packing kernel can be
# checked byte for byte.
PACK_KBLOCK = 64


# --------------------------------------------------------------------------- decode
def decode_f64(codes: np.ndarray, codebooks: np.ndarray) -> np.ndarray:
    """Eq. 4 (Sec. 2.4), restated as Eq. A3 (App. A.1), in float64.

    codes [N][G][M] integers, codebooks [M][2**B][g] -> W [N][G*g] float64.
    Group i of row n is sum over m of codeword C^(m)[codes[n, i, m]]; groups are
    concatenated along the row.  No intermediate rounding.
    """
    N, G, M = codes.shape
    Mc, _, g = codebooks.shape
    assert Mc == M
    C = codebooks.astype(np.float64)
    W = np.zeros((N, G, g), dtype=np.float64)
    for m in range(M):
        W += C[m][codes[:, :, m].astype(np.int64)]
    return W.reshape(N, G * g)


def decode_rule_f16(codes: np.ndarray, codebooks: np.ndarray) -> np.ndarray:
    """Eq. 4 under the fixed rounding rule of the decode kernel.

    The paper leaves the arithmetic of the sum open.  The rule: widen each
    fp16 codeword entry to fp32, add in ascending m with IEEE fp32 adds
    (round-to-nearest-even, subnormals kept), then round once to fp16 (RNE,
    overflow to +-inf).  Returns float16 [N][G*g].
    """
    N, G, M = codes.shape
    g = codebooks.shape[2]
    C = codebooks.astype(np.float32)
    acc = C[0][codes[:, :, 0].astype(np.int64)]
    for m in range(1, M):
        acc = (acc + C[m][codes[:, :, m].astype(np.int64)]).astype(np.float32)
    with np.errstate(over="ignore"):
        return acc.astype(np.float16).reshape(N, G * g)


def decode_kaq_f64(codes: np.ndarray, codebooks: np.ndarray) -> np.ndarray:
    """Kernel-aware grouping for 3x3 convs (Sec. 3.1.2; App. A.1 Eq. A4).

    One group = the h1*w1 taps of one (output channel, input channel) filter.
    codes [Cout][Cin][M], codebooks [M][2**B][h1*w1] -> F [Cout][Cin][h1*w1]
    (float64; reshape the last axis to (h1, w1), row-major taps).
    """
    Cout, Cin, M = codes.shape
    C = codebooks.astype(np.float64)
    F = np.zeros((Cout, Cin, C.shape[2]), dtype=np.float64)
    for m in range(M):
        F += C[m][codes[:, :, m].astype(np.int64)]
    return F


def kaq_ohwi(F: np.ndarray) -> np.ndarray:
    """Layout only: kernel-aware filters F [Cout][Cin][h1*w1] (taps row-major)
    -> the OHWI weight matrix [Cout][h1*w1*Cin] of ``conv2d_nhwc_f64``, reduction
    index k = t*Cin + c for tap t and input channel c."""
    Cout, Cin, taps = F.shape
    return np.ascontiguousarray(F.transpose(0, 2, 1)).reshape(Cout, taps * Cin)


def kaq_from_ohwi(W: np.ndarray, taps: int = 9) -> np.ndarray:
    """Layout only, the inverse of ``kaq_ohwi``: [Cout][taps*Cin] (k = t*Cin + c)
    -> [Cout][Cin][taps]."""
    Cout, K = W.shape
    Cin = K // taps
    return np.ascontiguousarray(W.reshape(Cout, taps, Cin).transpose(0, 2, 1))


def codebook_grad_f64(codes: np.ndarray, G: np.ndarray, scale: np.ndarray | None, s_x: float,
                      n_code: int) -> np.ndarray:
    """Backward of Eq. 4 with respect to the codebooks (the continuous step of
    Stage-2 fine-tuning, Sec. 3.2.1), float64.

    codes [N][Gr][M]; G [N][Gr*g] = dL/dW for the unscaled decoded weight, group i
    of row n at columns i*g .. i*g+g-1 (pass ``kaq_from_ohwi(G).reshape(N, -1)`` for
    the kernel-aware grouping).  The layer multiplies row n by s_x*scale[n], so
      dC[m][c][e] = sum over (n, i) with codes[n, i, m] == c of s_x*scale[n]*G[n][i*g+e].
    Returns dC [M][n_code][g].
    """
    N, Gr, M = codes.shape
    g = G.shape[1] // Gr
    f = float(s_x) * (scale.astype(np.float64) if scale is not None else np.ones(N))
    Gs = (G.astype(np.float64) * f[:, None]).reshape(N * Gr, g)
    dC = np.zeros((M, n_code, g), dtype=np.float64)
    for m in range(M):
        np.add.at(dC[m], codes[:, :, m].reshape(-1).astype(np.int64), Gs)
    return dC


def input_grad_f64(dy: np.ndarray, codes: np.ndarray, codebooks: np.ndarray,
                   scale: np.ndarray, alpha: float = 1.0) -> np.ndarray:
    """Backward of the layer with respect to its input (the gradient the continuous step of
    Sec. 3.2.1 passes to the layers before this one), float64.

    The layer of Sec. 3.1.1, Y = W X, with the decoded AQ weight of Eq. 4 and the
    per-output-channel scale: y[t, n] = scale[n] * sum_k X[t, k] * W[n, k] + bias[n],
    X = s_x * xq.  Its input gradient is
      dX[t, k] = sum_n dY[t, n] * scale[n] * W[n, k],
    returned times ``alpha`` (alpha = s_x: the gradient with respect to the codes xq).
    dy [T][N], codes [N][Gr][M], codebooks [M][2**B][g], scale [N] -> [T][Gr*g].
    """
    W = decode_f64(codes, codebooks)
    G = dy.astype(np.float64) * scale.astype(np.float64)[None, :]
    return float(alpha) * (G @ W)


def code_update_f32(W: np.ndarray, codebooks: np.ndarray, codes: np.ndarray,
                    H: np.ndarray | None = None, ms=None) -> np.ndarray:
    """One greedy code-search step (Stage-1 calibration, Sec. 3.1; the code
    optimisation of AQLM with beam width 1): for every group and each codebook m in
    ``ms`` in turn, replace code b[m] by the codeword that minimises the group's
    error with the other codebooks' codewords held fixed,
        r = w_group - sum_{m' != m} C^(m')[b[m']]          (ascending m')
        score(c) = d^T H d,  d = C^(m)[c] - r               (H = I when None)
    with H the group's g x g block of A A^T for calibration inputs A (the
    block-diagonal part of ||W A - W-hat A||^2).  The decision is taken in float32
    with a fixed operation order (each product and sum rounded separately,
    sums in ascending element index), ties to the lowest c.
    W [N][K] float32; codebooks [M][n_code][g]; codes [N][K/g][M] (a copy is
    updated and returned); H [K/g][g][g] float32 or None.  Pure Python loops over
    groups: small inputs only.
    """
    N, Gr, M = codes.shape
    Mc, n_code, g = codebooks.shape
    C = codebooks.astype(np.float32)
    Wf = W.astype(np.float32).reshape(N, Gr, g)
    out = codes.copy()
    ms = range(M) if ms is None else ms
    f32 = np.float32
    for n in range(N):
        for i in range(Gr):
            for m in ms:
                r = Wf[n, i].copy()
                for m2 in range(M):
                    if m2 != m:
                        r = (r - C[m2, int(out[n, i, m2])]).astype(f32)
                d = (C[m] - r[None, :]).astype(f32)               # [n_code][g]
                if H is None:
                    t = d
                else:
                    Hi = H[i].astype(f32)
                    t = np.zeros_like(d)
                    for e2 in range(g):
                        t = (t + (Hi[:, e2][None, :] * d[:, e2][:, None]).astype(f32)).astype(f32)
                score = np.zeros(n_code, dtype=f32)
                for e in range(g):
                    score = (score + (d[:, e] * t[:, e]).astype(f32)).astype(f32)
                out[n, i, m] = int(np.argmin(score))           # first minimum = lowest c
    return out


# --------------------------------------------------------------------------- packing
def packed_nbytes(N: int, K: int, g: int, M: int, B: int) -> int:
    """Bytes of the packed code buffer: ceil(K/64) blocks x N rows x (64/g) groups x M codes."""
    kblocks = -(-K // PACK_KBLOCK)
    return kblocks * N * (PACK_KBLOCK // g) * M * (B // 8)


def pack_codes(codes: np.ndarray, g: int) -> np.ndarray:
    """Packed storage order of the codes b[n, i, m] (a layout, not arithmetic).

    Canonical codes [N][K/g][M] are reordered to [K/64][N][64/g][M]: the codes
    that one output row needs for one 64-wide K block are contiguous (16 bytes
    for 2 codebooks of 8-bit codes), and consecutive rows are consecutive.  A
    K tail shorter than 64 is zero-padded.  uint16 codes are stored
    little-endian.  Returns the packed bytes as a flat uint8 array.
    """
    N, G, M = codes.shape
    per_block = PACK_KBLOCK // g
    kblocks = -(-G // per_block)
    out = np.zeros((kblocks, N, per_block, M), dtype=codes.dtype)
    for kb in range(kblocks):
        lo = kb * per_block
        hi = min(G, lo + per_block)
        out[kb, :, : hi - lo, :] = codes[:, lo:hi, :]
    return out.astype(codes.dtype.newbyteorder("<")).view(np.uint8).reshape(-1)


# --------------------------------------------------------------------------- activations
def quant_act(x: np.ndarray, s_x: float) -> np.ndarray:
    """8-bit activation quantizer (Sec. 4.2.3), the symmetric z = 0 form of Eq. 3.

    x_q = clip(round(x / s_x), -127, 127) with one scale per call (per
    timestep).  Reading of the paper: symmetric (no zero-point), the division
    x / s_x taken in IEEE fp32 (x is fp16, so widening is exact), round half to
    even, clip to [-127, 127] (-128 unused), NaN maps to 0.
    """
    # widening a signalling-NaN fp16 pattern raises the IEEE invalid flag; the value is
    # a NaN either way and maps to 0 below
    with np.errstate(invalid="ignore"):
        q = np.asarray(x).astype(np.float32) / np.float32(s_x)
    q = np.rint(q)
    q = np.where(np.isnan(q), np.float32(0.0), q)
    q = np.clip(q, -127.0, 127.0)
    return q.astype(np.int8)


# --------------------------------------------------------------------------- layers
def linear_f64(xq: np.ndarray, s_x: float, W: np.ndarray, scale: np.ndarray,
               bias: np.ndarray | None) -> np.ndarray:
    """Y = diag-scaled linear layer in float64 (Sec. 3.1.1: Y = W X).

    xq [T][K] int8, W [N][K] (decoded, float64), scale [N], bias [N] or None.
    Y[t, n] = scale[n] * sum_k (s_x * xq[t, k]) * W[n, k] + bias[n].
    """
    X = xq.astype(np.float64) * float(s_x)
    acc = X @ W.astype(np.float64).T
    y = acc * scale.astype(np.float64)[None, :]
    if bias is not None:
        y = y + bias.astype(np.float64)[None, :]
    return y


def conv2d_nhwc_f64(xq: np.ndarray, s_x: float, W: np.ndarray, scale: np.ndarray,
                    bias: np.ndarray | None, kh: int = 3, kw: int = 3,
                    stride: int = 1, pad: int = 1) -> np.ndarray:
    """Direct NHWC convolution in float64 (Sec. 3.1.1; App. A.1 Eq. A1).

    xq [Nb][H][W][Cin] int8, W [Cout][kh*kw*Cin] with reduction index
    k = (i*kw + j)*Cin + c (OHWI).  Zero padding `pad`, stride `stride`:
      Y[b, ho, wo, n] = scale[n] * sum_{i, j, c} s_x*xq[b, ho*s+i-pad, wo*s+j-pad, c]
                                           * W[n, (i*kw+j)*Cin + c]  + bias[n]
    with out-of-range input positions read as 0.  Summed tap by tap.
    """
    Nb, H, Wd, Cin = xq.shape
    Cout = W.shape[0]
    Wt = W.astype(np.float64).reshape(Cout, kh, kw, Cin)
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (Wd + 2 * pad - kw) // stride + 1
    Xp = np.zeros((Nb, H + 2 * pad, Wd + 2 * pad, Cin), dtype=np.float64)
    Xp[:, pad:pad + H, pad:pad + Wd, :] = xq.astype(np.float64) * float(s_x)
    acc = np.zeros((Nb, Ho, Wo, Cout), dtype=np.float64)
    for i in range(kh):
        for j in range(kw):
            patch = Xp[:, i:i + stride * (Ho - 1) + 1:stride,
                       j:j + stride * (Wo - 1) + 1:stride, :]
            acc += patch @ Wt[:, i, j, :].T
    y = acc * scale.astype(np.float64)
    if bias is not None:
        y = y + bias.astype(np.float64)
    return y


def lut_linear_f64(xq: np.ndarray, s_x: float, codes: np.ndarray,
                   codebooks: np.ndarray, scale: np.ndarray,
                   bias: np.ndarray | None) -> np.ndarray:
    """Lookup-table order of the same sum (App. A.1 Eq. A5 -> A6), float64.

    L[t, i, m, c] = sum_e x[t, i*g + e] * C^(m)[c, e]    (every codeword c)
    acc[t, n]     = sum_i sum_m L[t, i, m, b[n, i, m]]   (gather by code)
    Same value as decode-then-matmul up to rounding order.
    """
    T, K = xq.shape
    N, G, M = codes.shape
    g = codebooks.shape[2]
    X = xq.astype(np.float64).reshape(T, G, g) * float(s_x)
    C = codebooks.astype(np.float64)
    L = np.einsum("tie,mce->timc", X, C)
    acc = np.zeros((T, N), dtype=np.float64)
    gi = np.broadcast_to(np.arange(G)[None, :], (N, G))
    for m in range(M):
        acc += L[:, gi, m, codes[:, :, m].astype(np.int64)].sum(axis=-1)
    y = acc * scale.astype(np.float64)[None, :]
    if bias is not None:
        y = y + bias.astype(np.float64)[None, :]
    return y


def layer_f64(inp: dict) -> np.ndarray:
    """Reference output of an ``aq_synth`` layer dict (linear or conv).  A conv
    spec with g = 9 uses the kernel-aware grouping (Sec. 3.1.2): one group per
    (output channel, input channel) 3x3 filter."""
    spec = inp["spec"]
    if getattr(spec, "g", 8) == 9 and inp["xq"].ndim == 4:
        W = kaq_ohwi(decode_kaq_f64(inp["codes"], inp["codebooks"]))
    else:
        W = decode_f64(inp["codes"], inp["codebooks"])
    if inp["xq"].ndim == 2:
        return linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"])
    return conv2d_nhwc_f64(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"],
                           spec.kh, spec.kw, spec.stride, spec.pad)


# --------------------------------------------------------------------------- op counts
def lut_conv_kaq_counted(H: np.ndarray, codes: np.ndarray, codebooks: np.ndarray,
                         h1: int = 3, w1: int = 3):
    """The LUT inference kernel of App. A.1 (Eq. A6) with an operation counter.

    H [Cin][h][w] (one image, channels first), codes [Cout][Cin][M],
    codebooks [M][2**k][h1*w1].  Zero-padded 'same' convolution (the appendix
    pads so the spatial size is kept).  Step 1 convolves every input channel
    H_j with every codeword C^(m)_c; step 2 sums, for each output channel, the
    maps selected by its codes.  Counting follows Eq. A7: h1*w1 products and
    h1*w1 - 1 additions per output pixel of every (j, m, c) map, and one
    addition per selected map per output pixel (accumulation into zero).
    Returns (G [Cout][h][w] float64, mults, adds).  Pure Python loops: tiny
    inputs only.
    """
    Cin, h, w = H.shape
    Cout, _, M = codes.shape
    n_code = codebooks.shape[1]
    ph, pw = h1 // 2, w1 // 2
    mults = adds = 0
    # Step 1: table of maps H_j * C^(m)_c.
    maps = np.zeros((Cin, M, n_code, h, w), dtype=np.float64)
    for j in range(Cin):
        for m in range(M):
            for c in range(n_code):
                kern = codebooks[m, c].astype(np.float64).reshape(h1, w1)
                for y in range(h):
                    for x in range(w):
                        s = 0.0
                        first = True
                        for a in range(h1):
                            for b in range(w1):
                                yy, xx = y + a - ph, x + b - pw
                                v = float(H[j, yy, xx]) if (0 <= yy < h and 0 <= xx < w) else 0.0
                                p = v * float(kern[a, b])
                                mults += 1
                                if first:
                                    s = p
                                    first = False
                                else:
                                    s += p
                                    adds += 1
                        maps[j, m, c, y, x] = s
    # Step 2: gather-sum by code.
    G = np.zeros((Cout, h, w), dtype=np.float64)
    for i in range(Cout):
        for j in range(Cin):
            for m in range(M):
                sel = maps[j, m, int(codes[i, j, m])]
                for y in range(h):
                    for x in range(w):
                        G[i, y, x] += sel[y, x]
                        adds += 1
    return G, mults, adds


def direct_conv_counted(H: np.ndarray, F: np.ndarray):
    """Dense 'same' convolution with an operation counter (App. A.1 Eq. A2).

    H [Cin][h][w], F [Cout][Cin][h1][w1].  One multiply and one add per
    multiply-accumulate (the appendix's factor 2).  Returns (G, flops).
    """
    Cin, h, w = H.shape
    Cout, _, h1, w1 = F.shape
    ph, pw = h1 // 2, w1 // 2
    flops = 0
    G = np.zeros((Cout, h, w), dtype=np.float64)
    for i in range(Cout):
        for y in range(h):
            for x in range(w):
                s = 0.0
                for j in range(Cin):
                    for a in range(h1):
                        for b in range(w1):
                            yy, xx = y + a - ph, x + b - pw
                            v = float(H[j, yy, xx]) if (0 <= yy < h and 0 <= xx < w) else 0.0
                            s += v * float(F[i, j, a, b])
                            flops += 2
                G[i, y, x] = s
    return G, flops


def eq_a7_flops(M: int, k: int, Cin: int, Cout: int, h: int, w: int, h1: int = 3,
                w1: int = 3):
    """Eq. A7 (App. A.1): (multiplications, additions) of the LUT kernel."""
    mults = M * (2 ** k) * Cin * h * w * h1 * w1
    adds = M * (2 ** k) * Cin * h * w * (h1 * w1 - 1) + M * Cout * Cin * h * w
    return mults, adds


def eq_a2_flops(Cin: int, Cout: int, h: int, w: int, h1: int = 3, w1: int = 3) -> int:
    """Eq. A2 (App. A.1): FLOPs of a dense 'same' convolution."""
    return Cout * Cin * h * w * h1 * w1 * 2


def paper_lut_breakeven(M: int, k: int) -> float:
    """The break-even output-channel count printed at the end of App. A.1."""
    return 9 * (2 ** k - 1) * M / (2 * 9 - M)


def eq_a7_breakeven(M: int, k: int, h1: int = 3, w1: int = 3) -> float:
    """Smallest Cout at which Eq. A7 <= Eq. A2 (our re-derivation).

    M*Cin*hw*(2*h1*w1 - 1)*2**k + M*Cout*Cin*hw <= 2*h1*w1*Cout*Cin*hw
    <=>  Cout >= M * (2*h1*w1 - 1) * 2**k / (2*h1*w1 - M).
    """
    r = h1 * w1
    return M * (2 * r - 1) * (2 ** k) / (2 * r - M)


# --------------------------------------------------------------------------- storage
def bits_per_weight(codes: np.ndarray, codebooks: np.ndarray, scale: np.ndarray,
                    N: int, K: int) -> float:
    """Storage bits per weight measured from the actual buffers (Sec. 2.4).

    Codes are stored at their native width (uint8 for 8-bit codes, uint16 for
    16-bit codes), codebooks and scales in fp16.
    """
    return 8.0 * (codes.nbytes + codebooks.nbytes + scale.nbytes) / (N * K)


def bits_per_weight_closed_form(N: int, K: int, g: int, M: int, B: int) -> float:
    """M*B/g code bits + codebook overhead M*2**B*g*16/(N*K) + fp16 scale 16/K."""
    return M * B / g + M * (2 ** B) * g * 16 / (N * K) + 16 / K


# --------------------------------------------------------------------------- metrics
def compare(y: np.ndarray, y64: np.ndarray) -> dict:
    """Error metrics of an output against the float64 reference.

    rel_fro = ||y - y64||_F / ||y64||_F ; max_abs = max |y - y64| ;
    scale_ref = max |y64| (the max-abs bound is 1e-2 * scale_ref).
    Non-finite outputs make every metric infinite.
    """
    y = np.asarray(y, dtype=np.float64)
    if not np.all(np.isfinite(y)):
        return dict(rel_fro=math.inf, max_abs=math.inf, scale_ref=float(np.max(np.abs(y64))))
    d = y - y64
    nrm = float(np.linalg.norm(y64))
    return dict(rel_fro=float(np.linalg.norm(d) / nrm) if nrm > 0 else float(np.linalg.norm(d)),
                max_abs=float(np.max(np.abs(d))) if d.size else 0.0,
                scale_ref=float(np.max(np.abs(y64))) if y64.size else 0.0)
