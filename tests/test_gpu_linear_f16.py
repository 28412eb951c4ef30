"""GPU parity of aq_linear_f16 (the layer from fp16 activations in one call): the same
bits as aq_quant_act followed by aq_linear on every path and output type when both run
the same plan, and within tolerance of the fp64 oracle on the quantized activations."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_f16_activations, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack

pytestmark = pytest.mark.gpu

AUTO, DENSE, FUSED, LUT, FEW = 0, 1, 2, 3, 4


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _pair(inp, x16, s_x, path, out_f32):
    import torch
    import paper_2506_05960_gb300 as aq
    T, K = x16.shape
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    packed = pack(inp["codes"], N, K, M, B)
    books, scale, bias = dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"])
    dt = aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16
    tdt = torch.float32 if out_f32 else torch.float16
    x = dev(x16)
    # the two-call chain
    xq = torch.empty((T, K), dtype=torch.int8, device="cuda")
    aq.aq_quant_act(x, xq, T * K, s_x)
    wsb = aq.aq_linear_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    y_chain = torch.full((T, N), float("nan"), dtype=tdt, device="cuda")
    aq.aq_linear(xq, s_x, packed, books, scale, bias, y_chain, dt, T, K, N, 8, M, B, ws, wsb, path)
    # one call, on the chain's plan (on the dense paths aq_linear_f16 feeds the tensor cores
    # fp16 activations from shared memory and may choose another N tile or K split)
    pl = aq.aq_linear_plan(T, K, N, 8, M, B, path)
    if pl["BN"]:
        aq.aq_set_plan_override(pl["BN"], pl["splits"], pl["cluster"])
    try:
        pf = aq.aq_linear_f16_plan(T, K, N, 8, M, B, path)
        assert (pf["path"], pf["BN"], pf["splits"], pf["cluster"]) == (
            pl["path"], pl["BN"], pl["splits"], pl["cluster"])
        wsb2 = aq.aq_linear_f16_workspace_size(T, K, N, 8, M, B, path)
        assert wsb2 >= 2 * T * K
        ws2 = torch.full((wsb2,), 0x55, dtype=torch.uint8, device="cuda")
        y = torch.full((T, N), float("nan"), dtype=tdt, device="cuda")
        aq.aq_profile_enable(True)
        aq.aq_linear_f16(x, s_x, packed, books, scale, bias, y, dt, T, K, N, 8, M, B, ws2, wsb2,
                         path)
        torch.cuda.synchronize()
        prof = aq.aq_profile_read()
        aq.aq_profile_enable(False)
    finally:
        aq.aq_set_plan_override()
    assert aq.aq_device_error() == 0
    if pf["a16"]:   # the workspace holds the codes as fp16 values
        xq_ws = ws2[:2 * T * K].view(torch.float16).reshape(T, K)
        assert torch.equal(xq_ws, xq.to(torch.float16))
    else:           # the workspace holds the int8 codes
        xq_ws = ws2[:T * K].view(torch.int8).reshape(T, K)
        assert torch.equal(xq_ws, xq)
    return y.cpu().numpy(), y_chain.cpu().numpy(), xq.cpu().numpy(), prof


@pytest.mark.parametrize("T,K,N,M,B,path,out_f32", [
    (4096, 960, 2880, 2, 8, AUTO, False),      # the qkv projection: dense, quantizer + decode fused
    (300, 1024, 1152, 4, 8, DENSE, True),      # ragged row tile, fp32 output
    (1000, 512, 264, 1, 16, DENSE, False),     # 2^16 codebook decode in the same launch
    (128, 960, 960, 2, 8, AUTO, False),        # fused path (K split in cluster)
    (200, 208, 208, 2, 8, FUSED, True),        # ragged K block
    (3, 960, 2880, 2, 8, AUTO, False),         # few tokens
    (7, 576, 1728, 2, 8, LUT, False),          # table path
    (1, 64, 64, 2, 8, DENSE, False),           # one token
    (5, 80, 40, 2, 8, DENSE, True),            # one short ragged tile
])
def test_linear_f16_equals_chain(T, K, N, M, B, path, out_f32):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=T + K + N + M + path)
    x16 = make_f16_activations((T, K), seed=T + N, std=2.0)
    s_x = float(np.float32(0.05))                # exact ties of x / s_x for many fp16 values
    y, y_chain, xq, prof = _pair(inp, x16, s_x, path, out_f32)
    if out_f32:
        assert np.array_equal(y.view(np.uint32), y_chain.view(np.uint32))
    else:
        assert np.array_equal(y.view(np.uint16), y_chain.view(np.uint16))
    assert np.array_equal(xq, O.quant_act(x16, s_x))
    q_inp = dict(inp, xq=xq, s_x=s_x)
    assert_close(y.astype(np.float64), O.layer_f64(q_inp), (T, K, N, path))
    if path == DENSE or (path == AUTO and T >= 256):
        assert prof["quant"][1] == 1 and prof["decode"][1] == 1


def test_linear_f16_errors():
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=64, K=256, N=256, M=2, B=8), seed=3)
    packed = pack(inp["codes"], 256, 256, 2, 8)
    x = dev(make_f16_activations((64, 256), seed=1))
    y = torch.empty((64, 256), dtype=torch.float16, device="cuda")
    args = (x, 0.02, packed, dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"]), y,
            aq.AQ_DTYPE_F16, 64, 256, 256, 8, 2, 8)
    need = aq.aq_linear_f16_workspace_size(64, 256, 256, 8, 2, 8, DENSE)
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    with pytest.raises(aq.AQError) as e:                      # workspace too small
        aq.aq_linear_f16(*args, ws, need - 1024, DENSE)
    assert e.value.status == -5
    with pytest.raises(aq.AQError) as e:                      # s_x must be > 0
        aq.aq_linear_f16(x, 0.0, *args[2:], ws, need, DENSE)
    assert e.value.status == -2
    with pytest.raises(aq.AQError) as e:                      # int8 output: aq_linear_q8
        aq.aq_linear_f16(*args[:7], aq.AQ_DTYPE_I8, *args[8:], ws, need, DENSE)
    assert e.value.status == -3
    aq.aq_linear_f16(None, 0.02, None, None, None, None, None, aq.AQ_DTYPE_F16, 0, 256, 256, 8,
                     2, 8, None, 0, DENSE)                   # T == 0 is a no-op
