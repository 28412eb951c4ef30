"""GPU parity of the fused-decode path (weight tiles decoded into shared memory
inside the tensor-core kernel, W-hat never written to HBM) against the fp64
oracle, for linear and convolution layers and both code widths."""

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, ConvSpec, LinearSpec, make_conv, make_linear
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
    inp = make_conv(WORKLOADS["conv8_book16"], seed=SEEDS["conv8_book16"])
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


@pytest.mark.parametrize("path", [DENSE, FUSED])
@pytest.mark.parametrize("M,B", [(1, 8), (2, 8), (3, 8), (4, 8), (8, 8), (1, 16), (2, 16)])
def test_decode_inside_gemm_bit_exact(M, B, path):
    """Identity activations (x[t][k] = [t == k], s_x = scale = 1, no bias, fp32 out)
    make the layer return W-hat transposed exactly, so the weights the tensor core
    multiplied are compared bit for bit (as values: a zero's sign is not kept by
    the sum) with the decode rule of Eq. 4, on edge-value codebooks: subnormals,
    halfway cases, large magnitudes whose sums stay finite."""
    rng = np.random.default_rng(100 * M + B)
    K = 208                                 # ragged last K block (3.25 blocks)
    N = 72                                  # ragged N tile
    special = np.array([8000, -8000, 6e-8, -6e-8, 0.0, -0.0, 1.0, 2 ** -14, 1e-5,
                        1 + 2 ** -10, -(1 + 2 ** -10), 2049, 0.1, -3.0e-5], dtype=np.float16)
    books = special[rng.integers(0, special.size, size=(M, 1 << B, 8))].astype(np.float16)
    codes = rng.integers(0, 1 << B, size=(N, K // 8, M),
                         dtype=np.uint8 if B == 8 else np.uint16)
    inp = dict(xq=np.eye(K, dtype=np.int8), s_x=1.0, codebooks=books, codes=codes,
               scale=np.ones(N, dtype=np.float16), bias=np.zeros(N, dtype=np.float16))
    y = run_linear(inp, out_f32=True, with_bias=False, path=path)
    ref = O.decode_rule_f16(codes, books).astype(np.float64)      # [N][K]
    assert np.isfinite(ref).all()
    assert np.array_equal(y, ref.T)
