"""GPU parity of aq_conv2d_nhwc (implicit GEMM, 3x3, pad 1) against the fp64
oracle's direct convolution."""

import pytest

from aq_synth import SEEDS, WORKLOADS, ConvSpec, make_conv
from oracle import aq_oracle as O

from gpu_util import assert_close, run_conv

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("Nb,H,W,Cin,Cout,M", [
    (2, 8, 8, 64, 16, 2),       # two 8x8 images per 128-pixel tile
    (3, 8, 8, 64, 24, 2),       # ragged: last tile holds one image
    (1, 16, 16, 128, 64, 4),    # 8 rows of 16 per tile
    (2, 32, 32, 64, 200, 1),    # N tile tail
    (1, 64, 64, 64, 8, 2),      # 2 rows of 64 per tile
    (5, 4, 4, 64, 32, 2),       # 8 images per tile, ragged
])
def test_conv_shapes(Nb, H, W, Cin, Cout, M):
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, M=M, cb_std=0.05 / M ** 0.5)
    inp = make_conv(spec, seed=Nb * 1000 + H + Cin + Cout)
    y = run_conv(inp)
    assert_close(y, O.layer_f64(inp), spec)


@pytest.mark.parametrize("Nb,H,W,Cin,Cout,M", [
    (2, 64, 64, 192, 192, 2),   # UNet downsample 64 -> 32 (4 output rows per tile)
    (2, 16, 16, 64, 64, 4),     # 16 -> 8: two 8x8 output images per tile
    (3, 32, 32, 128, 96, 2),    # 32 -> 16, N tile tail
    (3, 16, 16, 576, 576, 2),   # UNet downsample 16 -> 8 at 576 channels, ragged images
])
def test_conv_stride2(Nb, H, W, Cin, Cout, M):
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, stride=2, M=M, cb_std=0.05 / M ** 0.5)
    inp = make_conv(spec, seed=7 * Nb + H + Cin)
    assert (spec.Ho, spec.Wo) == (H // 2, W // 2)
    y = run_conv(inp)
    assert_close(y, O.layer_f64(inp), spec)


def test_conv_fp32_no_bias():
    spec = ConvSpec(Nb=2, H=16, W=16, Cin=64, Cout=48, M=2)
    inp = make_conv(spec, seed=77)
    y = run_conv(inp, out_f32=True, with_bias=False)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y64 = O.conv2d_nhwc_f64(inp["xq"], inp["s_x"], W, inp["scale"], None)
    assert_close(y, y64)


def test_conv_64x64_w4a8_full():
    """16 x 64x64 x 192 -> 192, 4x8 codebooks: every output pixel and channel."""
    inp = make_conv(WORKLOADS["conv64"], seed=SEEDS["conv64"])
    y = run_conv(inp)
    assert_close(y, O.layer_f64(inp), "conv 64x64")


def test_conv_8x8_large_codebook_full():
    """2 x 8x8 x 960 -> 960, one 2^16-entry codebook (split-K plan)."""
    inp = make_conv(WORKLOADS["conv8_book16"], seed=SEEDS["conv8_book16"])
    y = run_conv(inp)
    assert_close(y, O.layer_f64(inp), "conv 8x8 1x16")
