"""GPU parity of aq_linear against the fp64 oracle (rel. Frobenius <= 2e-3,
max |err| <= 1e-2 * max|y64|), over the workload shapes, ragged tiles,
codebook formats, output dtypes and the split-K plan."""

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, LinearSpec, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, run_linear

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("out_f32", [False, True])
@pytest.mark.parametrize("with_bias", [True, False])
def test_tiny_linear_workload(out_f32, with_bias):
    inp = make_linear(WORKLOADS["tiny_linear"], seed=SEEDS["tiny_linear"])
    y = run_linear(inp, out_f32=out_f32, with_bias=with_bias)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y64 = O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], inp["bias"] if with_bias else None)
    assert_close(y, y64)


def test_qkv_projection_full():
    """T=4096, K=960, N=2880, 2x8 codebooks: every output against the oracle."""
    inp = make_linear(WORKLOADS["qkv"], seed=SEEDS["qkv"])
    y = run_linear(inp)
    assert_close(y, O.layer_f64(inp), "qkv")


@pytest.mark.parametrize("T,K,N", [(1, 64, 8), (5, 16, 24), (127, 208, 264), (129, 960, 512),
                                   (300, 1024, 1152), (64, 4096, 256), (2, 8640, 960)])
def test_ragged_and_split_shapes(T, K, N):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=2, B=8), seed=T + K + N)
    y = run_linear(inp)
    assert_close(y, O.layer_f64(inp), (T, K, N))


@pytest.mark.parametrize("M,B", [(1, 8), (3, 8), (4, 8), (8, 8), (1, 16), (2, 16)])
def test_codebook_formats(M, B):
    inp = make_linear(LinearSpec(T=200, K=320, N=136, M=M, B=B,
                                 cb_std=0.05 / np.sqrt(M)), seed=M * 10 + B)
    y = run_linear(inp, out_f32=True)
    assert_close(y, O.layer_f64(inp), (M, B))


def test_one_hot_books_exact():
    """One-hot books make W-hat an integer matrix: with s_x = scale = 1 and no bias the
    fp32 accumulation of |x| <= 127, |w| <= 128 over K = 512 is exact."""
    g = M = 8
    rng = np.random.default_rng(8)
    books = np.zeros((M, 256, g), dtype=np.float16)
    for m in range(M):
        books[m, :, m] = np.arange(256) - 128
    T, K, N = 130, 512, 40
    Wint = rng.integers(-128, 128, size=(N, K))
    codes = np.zeros((N, K // g, M), dtype=np.uint8)
    for m in range(M):
        codes[:, :, m] = (Wint[:, m::g] + 128).astype(np.uint8)
    xq = rng.integers(-127, 128, size=(T, K), dtype=np.int8)
    inp = dict(codebooks=books, codes=codes, scale=np.ones(N, np.float16),
               bias=np.zeros(N, np.float16), xq=xq, s_x=1.0, spec=None)
    y = run_linear(inp, out_f32=True)
    assert np.array_equal(y, (xq.astype(np.int64) @ Wint.T).astype(np.float64))
