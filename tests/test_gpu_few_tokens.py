"""GPU parity of the few-token path (linear layers with T <= 16 in one kernel: each
row's codes streamed once, decoded in registers, dotted with every token) against
the fp64 oracle, for every code format, ragged shapes and all output kinds."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, run_linear

pytestmark = pytest.mark.gpu

AUTO, FEW = 0, 4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("T", [1, 2, 3, 5, 8, 11, 16])
def test_few_tokens_qkv_shape(T):
    inp = make_linear(LinearSpec(T=T, K=960, N=2880, M=2, B=8), seed=T)
    y = run_linear(inp, path=FEW)
    assert_close(y, O.layer_f64(inp), T)
    if T <= 4:                                   # AUTO picks this path for a few tokens
        assert np.array_equal(run_linear(inp, path=AUTO), y)


@pytest.mark.parametrize("T,K,N,M,B", [
    (4, 256, 256, 1, 8), (7, 208, 40, 3, 8),         # ragged K block, N not a tile multiple
    (16, 512, 96, 8, 8), (2, 8640, 960, 1, 16),      # 8 codebooks; the 2^16-entry book
    (9, 1024, 24, 2, 16), (1, 17280, 960, 2, 8),      # long K (a 3x3 conv's im2col width)
])
def test_few_tokens_formats(T, K, N, M, B):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=T + K + N)
    assert_close(run_linear(inp, path=FEW), O.layer_f64(inp), (T, K, N, M, B))
    y32 = run_linear(inp, path=FEW, out_f32=True, with_bias=False)
    W = O.decode_f64(inp["codes"], inp["codebooks"])
    assert_close(y32, O.linear_f64(inp["xq"], inp["s_x"], W, inp["scale"], None))


@pytest.mark.parametrize("T,K,N,M", [(1, 8640, 960, 1), (1, 1024, 24, 2), (2, 8640, 960, 1),
                                     (4, 1024, 24, 2)])
def test_few_tokens_16bit_codes_at_auto_token_counts(T, K, N, M):
    """2^16-entry codebooks at the token counts AUTO sends down the few-token path
    (T <= 4): fp16 and fp32 outputs against the oracle, and AUTO gives the same bits."""
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=16, cb_std=0.05 / M ** 0.5),
                      seed=T * 7 + K + N)
    y = run_linear(inp, path=FEW)
    assert_close(y, O.layer_f64(inp), (T, K, N, M))
    assert np.array_equal(run_linear(inp, path=AUTO), y)
    y32 = run_linear(inp, path=FEW, out_f32=True)
    assert_close(y32, O.layer_f64(inp), (T, K, N, M, "f32"))
    assert np.array_equal(run_linear(inp, path=AUTO, out_f32=True), y32)


def test_few_tokens_q8_equals_chain():
    import torch
    import paper_2506_05960_gb300 as aq
    T, K, N, M, B = 6, 960, 2880, 2, 8
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B), seed=66)
    packed = pack(inp["codes"], N, K, M, B)
    args = (dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
            dev(inp["bias"]))
    y16 = torch.empty((T, N), dtype=torch.float16, device="cuda")
    aq.aq_linear(*args, y16, aq.AQ_DTYPE_F16, T, K, N, 8, M, B, None, 0, FEW)
    s_out = float(np.float32(0.8 * float(y16.abs().max()) / 127.0))
    q_chain = torch.empty((T, N), dtype=torch.int8, device="cuda")
    aq.aq_quant_act(y16, q_chain, T * N, s_out)
    q = torch.full((T, N), 99, dtype=torch.int8, device="cuda")
    aq.aq_linear_q8(*args, q, s_out, T, K, N, 8, M, B, None, 0, FEW)
    torch.cuda.synchronize()
    assert np.array_equal(q.cpu().numpy(), q_chain.cpu().numpy())


def test_few_tokens_refuses_more_tokens():
    import paper_2506_05960_gb300 as aq
    with pytest.raises(aq.AQError) as e:
        aq.aq_linear_workspace_size(17, 960, 960, 8, 2, 8, FEW)
    assert e.value.status == -3
