"""GPU parity of aq_linear_ex / aq_conv2d_nhwc_ex: the layer with the activation kind (int8
codes, or the codes held as fp16 values) and the output kind (fp16, fp32, the next layer's codes
under the activation rule of Sec. 4.2.3 as int8 or as fp16 values) as arguments.

Checks: the fp16-code output holds exactly the int8 output's codes on every path (dense, fused,
K split through the workspace or a cluster, few tokens, lookup table, convolution); fp16-code
input gives the same bits as int8 input under the same plan (the products of fp16 values are
exact and the K order is the same), and the layer tolerance against the fp64 oracle."""

import numpy as np
import pytest

from aq_synth import ConvSpec, LinearSpec, make_conv, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, poison

pytestmark = pytest.mark.gpu

AUTO, DENSE, FUSED, LUT, FEW, PRE = 0, 1, 2, 3, 4, 5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()
    yield
    aq.aq_set_plan_override()


def _linear(aq, inp, act_dtype, out_dtype, path=AUTO, s_out=0.05):
    import torch
    T, K = inp["xq"].shape
    N, _, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    packed = pack(inp["codes"], N, K, M, B)
    act = dev(inp["xq"] if act_dtype == aq.AQ_DTYPE_I8 else inp["xq"].astype(np.float16))
    wsb = aq.aq_linear_ex_workspace_size(act_dtype, T, K, N, 8, M, B, path)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    ydt = {aq.AQ_DTYPE_F16: torch.float16, aq.AQ_DTYPE_F32: torch.float32,
           aq.AQ_DTYPE_I8: torch.int8, aq.AQ_DTYPE_F16_CODES: torch.float16}[out_dtype]
    y = poison((T, N), ydt) if ydt != torch.int8 else torch.full((T, N), 99, dtype=ydt,
                                                                 device="cuda")
    aq.aq_linear_ex(act, act_dtype, inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
                    dev(inp["bias"]), y, out_dtype, s_out, T, K, N, 8, M, B, ws, wsb, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.cpu().numpy()


def _conv(aq, inp, act_dtype, out_dtype, path=AUTO, s_out=0.05):
    import torch
    s = inp["spec"]
    N, _, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    K = 9 * s.Cin
    packed = pack(inp["codes"], N, K, M, B, s.g)
    act = dev(inp["xq"] if act_dtype == aq.AQ_DTYPE_I8 else inp["xq"].astype(np.float16))
    args = (s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, 1, s.g, M, B, path)
    wsb = aq.aq_conv2d_ex_workspace_size(act_dtype, *args)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    shape = (s.Nb, s.Ho, s.Wo, s.Cout)
    ydt = {aq.AQ_DTYPE_F16: torch.float16, aq.AQ_DTYPE_F32: torch.float32,
           aq.AQ_DTYPE_I8: torch.int8, aq.AQ_DTYPE_F16_CODES: torch.float16}[out_dtype]
    y = poison(shape, ydt) if ydt != torch.int8 else torch.full(shape, 99, dtype=ydt,
                                                                device="cuda")
    aq.aq_conv2d_nhwc_ex(act, act_dtype, inp["s_x"], packed, dev(inp["codebooks"]),
                         dev(inp["scale"]), dev(inp["bias"]), y, out_dtype, s_out, *args[:12], ws,
                         wsb, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.cpu().numpy()


@pytest.mark.parametrize("T,K,N,M,B,path,override", [
    (4096, 960, 2880, 2, 8, AUTO, None),          # dense; both A forms below
    (128, 960, 960, 2, 8, AUTO, None),            # fused decode, K split in a cluster
    (300, 1024, 1152, 4, 8, DENSE, (128, 3, 0)),  # K split through the workspace + reduce
    (2, 960, 2880, 2, 8, AUTO, None),             # few tokens
    (8, 960, 2880, 2, 8, LUT, None),              # lookup-table path (reduce kernel)
    (2, 2048, 1040, 2, 8, LUT, None),             # rotated tables (chunk reduction)
    (3, 8640, 960, 1, 16, AUTO, None),            # few tokens, 2^16 codebook (gather kernel)
])
def test_code_outputs_agree(T, K, N, M, B, path, override):
    """fp16-code output == int8 output, element for element, on every path."""
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=T + K + N)
    s_out = float(np.float32(0.8 * np.abs(O.layer_f64(inp)).max() / 127.0))
    if override:
        aq.aq_set_plan_override(*override)
    try:
        q8 = _linear(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_I8, path, s_out)
        q16 = _linear(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_F16_CODES, path, s_out)
    finally:
        aq.aq_set_plan_override()
    assert np.array_equal(q16, q8.astype(np.float16))
    assert np.abs(q8.astype(np.int32)).max() > 64          # the codes span the range
    if path in (AUTO, DENSE) and T >= 128:
        # fp16 codes in, both output kinds: the shared-memory A form (dense paths)
        q16b = _linear(aq, inp, aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_F16_CODES, DENSE, s_out)
        q8b = _linear(aq, inp, aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_I8, DENSE, s_out)
        assert np.array_equal(q16b, q8b.astype(np.float16))
        # within one rounding step of the oracle's codes
        ref = O.quant_act(O.layer_f64(inp).astype(np.float16), s_out)
        assert np.abs(q8b.astype(np.int32) - ref.astype(np.int32)).max() <= 1


@pytest.mark.parametrize("T,K,N,M,B", [(4096, 960, 2880, 2, 8), (300, 1024, 264, 4, 8),
                                       (1000, 512, 1152, 1, 16)])
def test_f16_code_input_equals_int8_input_same_plan(T, K, N, M, B):
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5), seed=T + N)
    pl = aq.aq_linear_ex_plan(aq.AQ_DTYPE_I8, T, K, N, 8, M, B, DENSE)
    aq.aq_set_plan_override(pl["BN"], pl["splits"], pl["cluster"])
    try:
        y8 = _linear(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_F16, DENSE)
        pa = aq.aq_linear_ex_plan(aq.AQ_DTYPE_F16_CODES, T, K, N, 8, M, B, DENSE)
        assert pa["a16"] == 1 and (pa["BN"], pa["splits"]) == (pl["BN"], pl["splits"])
        ya = _linear(aq, inp, aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_F16, DENSE)
    finally:
        aq.aq_set_plan_override()
    assert np.array_equal(ya.view(np.uint16), y8.view(np.uint16))
    assert_close(ya.astype(np.float64), O.layer_f64(inp), (T, K, N))


@pytest.mark.parametrize("Nb,H,W,Cin,Cout,stride,M,g,path", [
    (16, 64, 64, 192, 192, 1, 4, 8, AUTO),   # the 64x64 W4A8 conv
    (2, 8, 8, 960, 960, 1, 2, 8, AUTO),      # fused path (int8 in), dense (fp16 codes in)
    (4, 32, 32, 128, 256, 2, 2, 8, AUTO),    # stride 2
    (2, 16, 16, 128, 256, 1, 2, 9, AUTO),    # kernel-aware g = 9
])
def test_conv_ex(Nb, H, W, Cin, Cout, stride, M, g, path):
    import paper_2506_05960_gb300 as aq
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, stride=stride, g=g, M=M,
                    cb_std=0.05 / M ** 0.5)
    inp = make_conv(spec, seed=Nb * H + Cin + Cout + g)
    y64 = O.layer_f64(inp)
    s_out = float(np.float32(0.8 * np.abs(y64).max() / 127.0))
    q8 = _conv(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_I8, path, s_out)
    q16 = _conv(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_F16_CODES, path, s_out)
    assert np.array_equal(q16, q8.astype(np.float16))
    # fp16 codes in (the shared-memory A form on a dense path), fp16 out: against the oracle,
    # and bit-equal to int8 in under the same plan
    ya = _conv(aq, inp, aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_F16, path)
    assert_close(ya.astype(np.float64), y64, spec)
    pl = aq.aq_conv2d_ex_plan(aq.AQ_DTYPE_I8, Nb, H, W, Cin, Cout, 3, 3, stride, 1, g, M, 8,
                              DENSE)
    aq.aq_set_plan_override(pl["BN"], pl["splits"], pl["cluster"])
    try:
        y8 = _conv(aq, inp, aq.AQ_DTYPE_I8, aq.AQ_DTYPE_F16, DENSE)
        yb = _conv(aq, inp, aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_F16, DENSE)
    finally:
        aq.aq_set_plan_override()
    assert np.array_equal(yb.view(np.uint16), y8.view(np.uint16))


def test_ex_errors():
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=64, K=256, N=256), seed=9)
    packed = pack(inp["codes"], 256, 256, 2, 8)
    books, scale = dev(inp["codebooks"]), dev(inp["scale"])
    xh = dev(inp["xq"].astype(np.float16))
    y = torch.empty((64, 256), dtype=torch.float16, device="cuda")
    wsb = aq.aq_linear_ex_workspace_size(aq.AQ_DTYPE_F16_CODES, 64, 256, 256, 8, 2, 8, AUTO)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    dims = (64, 256, 256, 8, 2, 8)
    with pytest.raises(aq.AQError) as e:                    # unknown activation kind
        aq.aq_linear_ex(xh, 7, 0.02, packed, books, scale, None, y, aq.AQ_DTYPE_F16, 0.0, *dims,
                        ws, wsb, AUTO)
    assert e.value.status == -3
    for path in (FUSED, LUT, FEW):                          # fp16 codes need a dense path
        with pytest.raises(aq.AQError) as e:
            aq.aq_linear_ex(xh, aq.AQ_DTYPE_F16_CODES, 0.02, packed, books, scale, None, y,
                            aq.AQ_DTYPE_F16, 0.0, *dims, ws, wsb, path)
        assert e.value.status == -3
    with pytest.raises(aq.AQError) as e:                    # code output needs s_out > 0
        aq.aq_linear_ex(xh, aq.AQ_DTYPE_F16_CODES, 0.02, packed, books, scale, None, y,
                        aq.AQ_DTYPE_F16_CODES, 0.0, *dims, ws, wsb, AUTO)
    assert e.value.status == -2
    xq = dev(inp["xq"])
    wsl = aq.aq_linear_workspace_size(64, 256, 256, 8, 2, 8, AUTO)
    wl = torch.empty(max(wsl, 16), dtype=torch.uint8, device="cuda")
    with pytest.raises(aq.AQError) as e:                    # fp16 codes out: only the _ex call
        aq.aq_linear(xq, 0.02, packed, books, scale, None, y, aq.AQ_DTYPE_F16_CODES, *dims, wl,
                     wsl, AUTO)
    assert e.value.status == -3
    aq.aq_linear_ex(None, aq.AQ_DTYPE_F16_CODES, 0.02, None, None, None, None, None,
                    aq.AQ_DTYPE_F16, 0.0, 0, 256, 256, 8, 2, 8, None, 0, AUTO)   # T == 0: no-op
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
