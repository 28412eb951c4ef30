"""GPU parity of the lookup-table path (App. A.1, Eq. A5-A6) of aq_linear
against the fp64 oracle, and its path-selection rules."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, run_linear

pytestmark = pytest.mark.gpu

LUT = 3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("T", [1, 2, 3, 4, 5, 8, 9, 16])
def test_lut_qkv_shape_small_batches(T):
    inp = make_linear(LinearSpec(T=T, K=960, N=2880, M=2, B=8), seed=100 + T)
    y = run_linear(inp, path=LUT)
    assert_close(y, O.layer_f64(inp), T)


@pytest.mark.parametrize("M", [1, 3, 4, 8])
@pytest.mark.parametrize("out_f32", [False, True])
def test_lut_codebook_counts(M, out_f32):
    inp = make_linear(LinearSpec(T=6, K=576, N=1728, M=M, B=8, cb_std=0.05 / M ** 0.5),
                      seed=200 + M)
    y = run_linear(inp, path=LUT, out_f32=out_f32)
    assert_close(y, O.layer_f64(inp), M)


def test_lut_ragged_k_and_no_bias():
    inp = make_linear(LinearSpec(T=7, K=208, N=40, M=2, B=8), seed=5)   # 26 groups
    y = run_linear(inp, path=LUT, with_bias=False)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    assert_close(y, O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], None))


def test_lut_matches_oracle_lut_order():
    """The kernel sums in the table order of Eq. A6; the oracle's table-order sum and its
    decode-order sum agree, and the GPU result is within tolerance of both."""
    inp = make_linear(LinearSpec(T=4, K=256, N=64, M=2, B=8), seed=9)
    y = run_linear(inp, path=LUT)
    y_lut = O.lut_linear_f64(inp["xq"], inp["s_x"], inp["codes"], inp["codebooks"],
                             inp["scale"], inp["bias"])
    assert_close(y, y_lut)


def test_lut_path_selection():
    import paper_2506_05960_gb300 as aq
    # AUTO takes the few-token path (no workspace) up to 4 tokens, the tensor-core path
    # beyond; the table path is taken on request
    assert aq.aq_linear_workspace_size(4, 960, 2880, 8, 2, 8, 0) == 0
    assert aq.aq_linear_workspace_size(8, 960, 2880, 8, 2, 8, LUT) > 0
    assert aq.aq_linear_workspace_size(256, 960, 2880, 8, 2, 8, 0) == \
        aq.aq_linear_workspace_size(256, 960, 2880, 8, 2, 8, 1)
    with pytest.raises(aq.AQError) as e:
        aq.aq_linear_workspace_size(4, 960, 960, 8, 1, 16, LUT)      # 2^16 codebook
    assert e.value.status == -3
    with pytest.raises(aq.AQError) as e:
        aq.aq_linear_workspace_size(17, 960, 960, 8, 2, 8, LUT)      # too many tokens
    assert e.value.status == -3


@pytest.mark.parametrize("T,K,N,M", [
    (1, 960, 2880, 2),       # the qkv projection
    (1, 208, 40, 2),         # 26 groups: the last packed K block half empty; N not a warp multiple
    (1, 4096, 4096, 2),      # many chunks and row slices
    (1, 576, 1728, 1),       # one codebook: 8 K blocks per chunk
    (1, 576, 1736, 3),       # three codebooks (general index arithmetic)
    (1, 1024, 512, 4),
    (1, 512, 264, 5),
    (1, 640, 96, 8),         # one K block per chunk
    (2, 960, 2880, 2),       # two floats per entry
    (2, 208, 40, 1),
    (2, 1024, 520, 4),
    (3, 960, 2880, 2),       # four floats per entry, one token unused
    (4, 4096, 4096, 2),
    (4, 208, 264, 1),
    (4, 1024, 512, 4),       # a chunk is a quarter of a packed record
    (1, 8192, 4104, 2),      # 129 CTAs whose row-block ranges cross chunk boundaries; 8-row tail
    (2, 4096, 1032, 1),
])
def test_lut_vector_tables(T, K, N, M):
    """Up to four tokens: the rotated-table kernel (M = 1, 2 or 4; 1, 2 or 4 floats per entry)
    and the one-token kernel for other M, against the oracle's decode order and table order, fp16
    and fp32 outputs."""
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=8, cb_std=0.05 / M ** 0.5),
                      seed=300 + T + K + N + M)
    ref = O.layer_f64(inp)
    assert_close(run_linear(inp, path=LUT), ref, (K, N, M))
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y32 = run_linear(inp, path=LUT, out_f32=True, with_bias=False)
    assert_close(y32, O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], None), (K, N, M))
    y_lut = O.lut_linear_f64(inp["xq"], inp["s_x"], inp["codes"], inp["codebooks"],
                             inp["scale"], inp["bias"])
    assert_close(run_linear(inp, path=LUT), y_lut, "table order")
    assert aq.aq_linear_workspace_size(T, K, N, 8, M, 8, LUT) > 0


@pytest.mark.parametrize("T,K,N,M", [(1, 16, 8, 2), (2, 64, 8, 1), (4, 16, 8, 4), (3, 32, 24, 2)])
def test_lut_smallest_layers(T, K, N, M):
    """The smallest layers the table path takes: one partial packed record, one partial row
    block, a single CTA; against the oracle in both output types."""
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=8, cb_std=0.05 / M ** 0.5),
                      seed=900 + T + K + N + M)
    assert_close(run_linear(inp, path=LUT), O.layer_f64(inp), (T, K, N, M))
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    y32 = run_linear(inp, path=LUT, out_f32=True, with_bias=False)
    assert_close(y32, O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], None), (T, K, N, M))

