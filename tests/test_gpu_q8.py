"""GPU parity of the layers whose epilogue writes the next layer's 8-bit
activations (aq_linear_q8 / aq_conv2d_nhwc_q8): bit-exact against the unfused
chain -- the same layer with fp16 output, then aq_quant_act with the same scale
-- on every execution path, and within one quantization step of the fp64
oracle's output passed through the quantizer rule."""

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, ConvSpec, LinearSpec, make_conv, make_linear
from oracle import aq_oracle as O

from gpu_util import dev, pack

pytestmark = pytest.mark.gpu

AUTO, DENSE, FUSED, LUT = 0, 1, 2, 3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _s_out(y64):
    # a scale that clips the largest outputs, so clipping is exercised too
    return float(np.float32(0.8 * np.abs(y64).max() / 127.0))


def _check(q, q_chain, y64, s_out):
    assert np.array_equal(q, q_chain)
    ref = O.quant_act(y64.astype(np.float16), s_out)
    assert np.abs(q.astype(np.int32) - ref.astype(np.int32)).max() <= 1


def _linear_pair(inp, path, s_out=None):
    import torch
    import paper_2506_05960_gb300 as aq
    xq = inp["xq"]
    T, K = xq.shape
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    packed = pack(inp["codes"], N, K, M, B)
    ws_bytes = aq.aq_linear_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    args = (dev(xq), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"]))
    y16 = torch.empty((T, N), dtype=torch.float16, device="cuda")
    aq.aq_linear(*args, y16, aq.AQ_DTYPE_F16, T, K, N, 8, M, B, ws, ws_bytes, path)
    y64 = O.layer_f64(inp)
    if s_out is None:
        s_out = _s_out(y64)
    q_chain = torch.empty((T, N), dtype=torch.int8, device="cuda")
    aq.aq_quant_act(y16, q_chain, T * N, s_out)
    q = torch.full((T, N), 99, dtype=torch.int8, device="cuda")
    aq.aq_linear_q8(*args, q, s_out, T, K, N, 8, M, B, ws, ws_bytes, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return q.cpu().numpy(), q_chain.cpu().numpy(), y64, s_out


@pytest.mark.parametrize("T,K,N,M,B,path", [
    (4096, 960, 2880, 2, 8, AUTO),     # the qkv projection, dense path
    (300, 1024, 1152, 4, 8, DENSE),    # ragged M tile
    (200, 208, 208, 2, 8, FUSED),      # ragged K block and N tile
    (128, 8640, 960, 1, 16, AUTO),     # 2^16 book, fused with split K (reduce epilogue)
    (5, 960, 2880, 2, 8, AUTO),        # fused path, one ragged row tile
    (1, 4096, 4112, 2, 8, LUT),        # rotated tables, 32 chunks (chunk reduction epilogue)
    (3, 2048, 1040, 4, 8, LUT),        # four floats per entry, a chunk is part of a record
    (4, 1024, 528, 1, 8, LUT),
    (6, 960, 2880, 2, 8, LUT),         # the general table kernel (split reduction epilogue)
])
def test_linear_q8_equals_chain(T, K, N, M, B, path):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=T + K + N + M + path)
    _check(*_linear_pair(inp, path))


@pytest.mark.parametrize("s_out", [0.05, 0.125, 0.02, 0.0473])
@pytest.mark.parametrize("path", [DENSE, FUSED])
def test_linear_q8_scales_with_exact_ties(s_out, path):
    """Scales with few significant bits make x / s_out an exact half-integer for many
    fp16 outputs (0.05 at x = 0.875): the epilogue's exact tie handling must still give
    the chain's bits."""
    inp = make_linear(LinearSpec(T=512, K=512, N=1024, M=2, B=8, cb_std=0.05 / 2 ** 0.5),
                      seed=int(s_out * 1e4) + path)
    q, q_chain, y64, s = _linear_pair(inp, path, s_out=float(np.float32(s_out)))
    assert np.array_equal(q, q_chain)


@pytest.mark.parametrize("wl,path", [("conv64", AUTO), ("conv8_book16", AUTO)])
def test_conv_q8_equals_chain(wl, path):
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_conv(WORKLOADS[wl], seed=SEEDS[wl])
    s = inp["spec"]
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    K = 9 * s.Cin
    packed = pack(inp["codes"], N, K, M, B)
    ws_bytes = aq.aq_conv2d_workspace_size(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, 1, 8,
                                           M, B, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    args = (dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
            dev(inp["bias"]))
    geo = (s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, 1, 8, M, B, ws, ws_bytes, path)
    shape = (s.Nb, s.Ho, s.Wo, s.Cout)
    y16 = torch.empty(shape, dtype=torch.float16, device="cuda")
    aq.aq_conv2d_nhwc(*args, y16, aq.AQ_DTYPE_F16, *geo)
    y64 = O.layer_f64(inp)
    s_out = _s_out(y64)
    q_chain = torch.empty(shape, dtype=torch.int8, device="cuda")
    aq.aq_quant_act(y16, q_chain, y16.numel(), s_out)
    q = torch.full(shape, 99, dtype=torch.int8, device="cuda")
    aq.aq_conv2d_nhwc_q8(*args, q, s_out, *geo)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    _check(q.cpu().numpy(), q_chain.cpu().numpy(), y64, s_out)


def test_q8_argument_errors():
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=64, K=256, N=264, M=2, B=8), seed=5)
    packed = pack(inp["codes"], 264, 256, 2, 8)
    ws_bytes = aq.aq_linear_workspace_size(64, 256, 264, 8, 2, 8, DENSE)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    q = torch.empty((64, 264), dtype=torch.int8, device="cuda")
    args = (dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
            dev(inp["bias"]), q)
    with pytest.raises(aq.AQError):          # N % 16 != 0
        aq.aq_linear_q8(*args, 0.1, 64, 256, 264, 8, 2, 8, ws, ws_bytes, DENSE)
    with pytest.raises(aq.AQError):          # s_out must be > 0
        aq.aq_linear_q8(*args, 0.0, 64, 256, 256, 8, 2, 8, ws, ws_bytes, DENSE)
    with pytest.raises(aq.AQError):          # int8 output only through the _q8 entry point
        aq.aq_linear(*args, aq.AQ_DTYPE_I8, 64, 256, 256, 8, 2, 8, ws, ws_bytes, DENSE)
