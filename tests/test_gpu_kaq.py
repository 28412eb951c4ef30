"""GPU parity of the kernel-aware grouping (Sec. 3.1.2; App. A.1 Eq. A4): one AQ
group per (output channel, input channel) 3x3 filter, g = 9.  The decode is
bit-exact against the rule (fp32 sum in ascending m, one RNE to fp16) written in
the convolution's OHWI order; the conv layer matches the fp64 oracle."""

import numpy as np
import pytest

from aq_synth import ConvSpec, make_conv
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, run_conv

pytestmark = pytest.mark.gpu

DENSE, FUSED = 1, 2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _books(rng, M, B, edge):
    if not edge:
        return rng.normal(0, 0.05, size=(M, 1 << B, 9)).astype(np.float16)
    special = np.array([65504, -65504, 32768, 6e-8, -6e-8, 0.0, -0.0, 1.0, 2 ** -14, 1e-5,
                        1 + 2 ** -10, 0.1], dtype=np.float16)
    return special[rng.integers(0, special.size, size=(M, 1 << B, 9))].astype(np.float16)


@pytest.mark.parametrize("M,B,edge", [(1, 8, True), (2, 8, True), (3, 8, True), (4, 8, False),
                                      (8, 8, True), (1, 16, False), (2, 16, True)])
def test_decode_kaq_bit_exact(M, B, edge):
    import torch
    import paper_2506_05960_gb300 as aq
    rng = np.random.default_rng(10 * M + B)
    Cout, Cin = 40, 37                       # ragged: nothing is a multiple of a tile
    books = _books(rng, M, B, edge)
    codes = rng.integers(0, 1 << B, size=(Cout, Cin, M), dtype=np.uint8 if B == 8 else np.uint16)
    codes[0] = 0
    codes[1] = (1 << B) - 1
    K = 9 * Cin
    packed = pack(codes, Cout, K, M, B, g=9)
    assert np.array_equal(packed.cpu().numpy().view(codes.dtype).reshape(codes.shape), codes)
    W = torch.full((Cout, K), float("nan"), dtype=torch.float16, device="cuda")
    aq.aq_decode(packed, dev(books), W, Cout, K, 9, M, B)
    rule = O.decode_rule_f16(codes, books).reshape(Cout, Cin, 9)      # [n][c][tap]
    ref = O.kaq_ohwi(rule.astype(np.float32)).astype(np.float16)       # [n][tap*Cin + c]
    assert np.array_equal(W.cpu().numpy().view(np.uint16), ref.view(np.uint16))


@pytest.mark.parametrize("Nb,H,W,Cin,Cout,stride,M,B", [
    (2, 8, 8, 64, 16, 1, 2, 8),        # two images per 128-pixel tile
    (1, 16, 16, 128, 64, 1, 4, 8),     # 8 rows of 16 per tile
    (2, 32, 32, 64, 200, 1, 2, 8),     # N tile tail
    (3, 16, 16, 64, 64, 2, 2, 8),      # stride 2
    (2, 8, 8, 192, 96, 1, 1, 16),      # 2^16-entry codebook, split K
])
def test_conv_kaq(Nb, H, W, Cin, Cout, stride, M, B):
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, stride=stride, g=9, M=M, B=B,
                    cb_std=0.05 / M ** 0.5)
    inp = make_conv(spec, seed=500 + Nb * H + Cin + Cout)
    assert inp["codes"].shape == (Cout, Cin, M) and inp["codebooks"].shape[2] == 9
    y = run_conv(inp)                       # AUTO: the dense path
    assert_close(y, O.layer_f64(inp), spec)
    yd = run_conv(inp, path=DENSE, out_f32=True)
    assert_close(yd, O.layer_f64(inp), spec)


def test_conv_kaq_fused_path_is_refused():
    import paper_2506_05960_gb300 as aq
    spec = ConvSpec(Nb=1, H=8, W=8, Cin=64, Cout=16, g=9, M=2)
    inp = make_conv(spec, seed=1)
    with pytest.raises(aq.AQError):
        run_conv(inp, path=FUSED)
