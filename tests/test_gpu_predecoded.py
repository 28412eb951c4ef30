"""GPU parity of AQ_PATH_PREDECODED: the dense path's GEMM on a workspace whose W-hat
was written beforehand by aq_decode (e.g. on another stream) gives the same bits as
the dense path with its own decode, for linear and 3x3 conv layers (g = 8 and the
kernel-aware g = 9), fp16/fp32/int8 outputs and the fp16-input entry point."""

import numpy as np
import pytest

from aq_synth import ConvSpec, LinearSpec, make_conv, make_f16_activations, make_linear

from gpu_util import dev, pack

pytestmark = pytest.mark.gpu

DENSE, PRE = 1, 5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("T,K,N,M,B,out", [
    (4096, 960, 2880, 2, 8, "f16"),
    (300, 1024, 1152, 4, 8, "f32"),
    (1000, 512, 264, 1, 16, "f16"),
    (600, 256, 512, 2, 8, "q8"),
])
def test_linear_predecoded_equals_dense(T, K, N, M, B, out):
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5), seed=T + N)
    packed = pack(inp["codes"], N, K, M, B)
    books, scale, bias, xq = (dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"]),
                              dev(inp["xq"]))
    wsb = aq.aq_linear_workspace_size(T, K, N, 8, M, B, DENSE)
    assert aq.aq_linear_workspace_size(T, K, N, 8, M, B, PRE) == wsb
    res = {}
    for path in (DENSE, PRE):
        ws = torch.full((wsb,), 0x7F, dtype=torch.uint8, device="cuda")
        if path == PRE:
            aq.aq_decode(packed, books, ws, N, K, 8, M, B)       # W-hat at the workspace start
        if out == "q8":
            y = torch.empty((T, N), dtype=torch.int8, device="cuda")
            aq.aq_linear_q8(xq, inp["s_x"], packed, books, scale, bias, y, 0.05, T, K, N, 8, M,
                            B, ws, wsb, path)
        else:
            y = torch.empty((T, N), dtype=torch.float32 if out == "f32" else torch.float16,
                            device="cuda")
            aq.aq_linear(xq, inp["s_x"], packed, books, scale, bias, y,
                         aq.AQ_DTYPE_F32 if out == "f32" else aq.AQ_DTYPE_F16, T, K, N, 8, M, B,
                         ws, wsb, path)
        torch.cuda.synchronize()
        assert aq.aq_device_error() == 0
        res[path] = y.cpu()
    assert torch.equal(res[DENSE].view(torch.uint8), res[PRE].view(torch.uint8))


@pytest.mark.parametrize("g", [8, 9])
def test_conv_predecoded_equals_dense(g):
    import torch
    import paper_2506_05960_gb300 as aq
    s = ConvSpec(Nb=2, H=16, W=16, Cin=192, Cout=200, g=g, M=2, B=8)
    inp = make_conv(s, seed=g)
    N, K = s.Cout, 9 * s.Cin
    packed = pack(inp["codes"], N, K, 2, 8, g)
    books, scale, bias, xq = (dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"]),
                              dev(inp["xq"]))
    wsb = aq.aq_conv2d_workspace_size(2, 16, 16, 192, 200, 3, 3, 1, 1, g, 2, 8, DENSE)
    res = {}
    for path in (DENSE, PRE):
        ws = torch.full((wsb,), 0x7F, dtype=torch.uint8, device="cuda")
        if path == PRE:
            aq.aq_decode(packed, books, ws, N, K, g, 2, 8)
        y = torch.empty((2, 16, 16, 200), dtype=torch.float16, device="cuda")
        aq.aq_conv2d_nhwc(xq, inp["s_x"], packed, books, scale, bias, y, aq.AQ_DTYPE_F16, 2, 16,
                          16, 192, 200, 3, 3, 1, 1, g, 2, 8, ws, wsb, path)
        torch.cuda.synchronize()
        assert aq.aq_device_error() == 0
        res[path] = y.cpu()
    assert torch.equal(res[DENSE].view(torch.int16), res[PRE].view(torch.int16))


def test_linear_f16_predecoded():
    import torch
    import paper_2506_05960_gb300 as aq
    T, K, N = 512, 960, 960
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=2, B=8), seed=77)
    packed = pack(inp["codes"], N, K, 2, 8)
    books, scale, bias = dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"])
    x = dev(make_f16_activations((T, K), seed=5, std=2.0))
    res = {}
    for path in (DENSE, PRE):
        wsb = aq.aq_linear_f16_workspace_size(T, K, N, 8, 2, 8, path)
        ws = torch.zeros(wsb, dtype=torch.uint8, device="cuda")
        if path == PRE:
            off = (2 * T * K + 1023) // 1024 * 1024        # W-hat follows the activation codes
            aq.aq_decode(packed, books, ws[off:], N, K, 8, 2, 8)
        y = torch.empty((T, N), dtype=torch.float16, device="cuda")
        aq.aq_linear_f16(x, 0.05, packed, books, scale, bias, y, aq.AQ_DTYPE_F16, T, K, N, 8, 2,
                         8, ws, wsb, path)
        torch.cuda.synchronize()
        res[path] = y.cpu()
    assert torch.equal(res[DENSE].view(torch.int16), res[PRE].view(torch.int16))
