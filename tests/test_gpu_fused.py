"""GPU parity of the fused-decode path (weight tiles decoded into shared memory
inside the tensor-core kernel, W-hat never written to HBM) against the fp64
oracle, for linear and convolution layers and both code widths."""

import numpy as np
import pytest

from aq_synth import CONFIGS, ConvSpec, LinearSpec, make_conv, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, run_conv, run_linear

pytestmark = pytest.mark.gpu

DENSE, FUSED = 1, 2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("T,K,N,M,B", [
    (64, 256, 256, 2, 8),       # tiny workload
    (5, 64, 24, 3, 8),
    (200, 208, 200, 2, 8),      # ragged K block, ragged N tile, 2 M tiles
    (300, 1024, 1152, 4, 8),
    (128, 8640, 960, 1, 16),    # 2^16-entry codebook gathered from L2, split K
    (33, 960, 2880, 2, 16),
])
def test_fused_linear(T, K, N, M, B):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=T * 7 + K + N + M)
    y = run_linear(inp, path=FUSED)
    assert_close(y, O.layer_f64(inp), (T, K, N, M, B))


def test_fused_linear_fp32_matches_dense():
    inp = make_linear(LinearSpec(T=100, K=512, N=384, M=2, B=8), seed=42)
    yf = run_linear(inp, path=FUSED, out_f32=True)
    yd = run_linear(inp, path=DENSE, out_f32=True)
    y64 = O.layer_f64(inp)
    assert_close(yf, y64)
    assert_close(yd, y64)
    # both paths multiply the same bit-exact fp16 weights: they agree to fp32 round-off
    np.testing.assert_allclose(yf, yd, rtol=1e-5, atol=1e-5 * np.abs(y64).max())


def test_fused_conv_large_codebook_full():
    """2 x 8x8 x 960 -> 960, one 2^16-entry codebook: the fused path with split K."""
    inp = make_conv(CONFIGS[3], seed=3)
    y = run_conv(inp, path=FUSED)
    assert_close(y, O.layer_f64(inp), "conv 8x8 1x16 fused")


@pytest.mark.parametrize("stride", [1, 2])
def test_fused_conv_small(stride):
    spec = ConvSpec(Nb=2, H=16, W=16, Cin=128, Cout=64, stride=stride, M=2)
    inp = make_conv(spec, seed=11 + stride)
    y = run_conv(inp, path=FUSED)
    assert_close(y, O.layer_f64(inp), spec)


def test_auto_paths_small_tokens_run_fused_or_lut():
    import paper_2506_05960_gb300 as aq
    # one M tile: AUTO decodes inside the GEMM (no W-hat in the workspace)
    assert aq.aq_linear_workspace_size(128, 960, 2880, 8, 2, 8, 0) == \
        aq.aq_linear_workspace_size(128, 960, 2880, 8, 2, 8, FUSED)
    assert aq.aq_linear_workspace_size(128, 960, 2880, 8, 2, 8, FUSED) < 960 * 2880 * 2
