"""GPU parity of aq_conv2d_nhwc_f16: the 8-bit activation quantizer (Sec. 4.2.3) and the 3x3
NHWC convolution (Sec. 3.1.1, implicit GEMM) in one call from fp16 activations.

When the shared-memory A form's plan has no K split and a wider N tile than the int8 form's
(or a plan override asks for a tile wider than 192), the codes are kept in the workspace as fp16
values and read through 4-D NHWC TMA boxes with the 128-byte swizzle.  Otherwise the call
quantizes to int8 for the tensor-memory A form, and then gives the same bits as aq_quant_act
followed by aq_conv2d_nhwc.  Every output is checked against the fp64 oracle on the
oracle's own quantization of the same fp16 activations."""

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, ConvSpec, make_conv, make_f16_activations
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, poison, run_conv

pytestmark = pytest.mark.gpu

AUTO, DENSE = 0, 1


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()
    yield
    aq.aq_set_plan_override()


def _run(inp, x16, s_x, path=AUTO, out_f32=False, with_bias=True):
    import torch
    import paper_2506_05960_gb300 as aq
    s = inp["spec"]
    N, _, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    K = s.kh * s.kw * s.Cin
    packed = pack(inp["codes"], N, K, M, B, s.g)
    args = (s.Nb, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw, s.stride, s.pad, s.g, M, B, path)
    plan = aq.aq_conv2d_f16_plan(*args)
    wsb = aq.aq_conv2d_f16_workspace_size(*args)
    ws = torch.full((wsb,), 0x55, dtype=torch.uint8, device="cuda")
    y = poison((s.Nb, s.Ho, s.Wo, s.Cout), torch.float32 if out_f32 else torch.float16)
    aq.aq_conv2d_nhwc_f16(dev(x16), s_x, packed, dev(inp["codebooks"]), dev(inp["scale"]),
                          dev(inp["bias"]) if with_bias else None, y,
                          aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, s.Nb, s.H, s.W, s.Cin,
                          s.Cout, s.kh, s.kw, s.stride, s.pad, s.g, M, B, ws, wsb, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.float().cpu().numpy().astype(np.float64), ws, plan


def _activations(spec, seed):
    x16 = make_f16_activations((spec.Nb, spec.H, spec.W, spec.Cin), seed=seed, std=2.0)
    s_x = float(np.float32(0.02))
    return x16, s_x, O.quant_act(x16, s_x)


def _check_codes(ws, plan, xq):
    """The quantized activations at the start of the workspace: fp16 values of the codes for
    the shared-memory A form, int8 codes otherwise (the oracle's quantizer rule either way)."""
    import torch
    n = xq.size
    if plan["a16"]:
        codes = ws[: 2 * n].view(torch.float16).cpu().numpy().reshape(xq.shape)
        assert np.array_equal(codes, xq.astype(np.float16))
    else:
        codes = ws[:n].view(torch.int8).cpu().numpy().reshape(xq.shape)
        assert np.array_equal(codes, xq)


@pytest.mark.parametrize("Nb,H,W,Cin,Cout,stride,M,B,g,override,path", [
    (16, 32, 32, 128, 256, 1, 2, 8, 8, None, AUTO),      # the planner's own fp16-form plan
    (4, 32, 32, 128, 256, 1, 2, 8, 8, (256, 1, 0), AUTO),  # one 256-wide tile, no K split
    (4, 32, 32, 128, 256, 1, 2, 8, 8, (256, 3, 1), AUTO),  # K split summed in a cluster
    (4, 32, 32, 128, 256, 1, 2, 8, 8, (256, 2, 0), AUTO),  # K split through the workspace
    (2, 32, 32, 192, 384, 2, 2, 8, 8, (256, 1, 0), AUTO),  # stride 2, ragged second N tile
    (3, 32, 32, 64, 264, 1, 2, 8, 8, (256, 1, 0), AUTO),   # N tail of 8 channels
    (2, 16, 16, 128, 256, 1, 2, 8, 9, (256, 1, 0), AUTO),  # kernel-aware g = 9
    (4, 16, 16, 64, 224, 1, 1, 16, 8, (224, 1, 0), DENSE),  # one 2^16-entry codebook
    (5, 4, 4, 64, 256, 1, 2, 8, 8, (256, 1, 0), DENSE),    # 8 images per 128-pixel tile, ragged
])
def test_conv_f16_shared_memory_a(Nb, H, W, Cin, Cout, stride, M, B, g, override, path):
    import paper_2506_05960_gb300 as aq
    spec = ConvSpec(Nb=Nb, H=H, W=W, Cin=Cin, Cout=Cout, stride=stride, g=g, M=M, B=B,
                    cb_std=0.05 / M ** 0.5)
    inp = make_conv(spec, seed=900 + Nb * H + Cin + Cout + g)
    x16, s_x, xq = _activations(spec, seed=Nb + H + Cout)
    if override:
        aq.aq_set_plan_override(*override)
    try:
        y, ws, plan = _run(inp, x16, s_x, path)
        y32, _, _ = _run(inp, x16, s_x, path, out_f32=True, with_bias=False)
    finally:
        aq.aq_set_plan_override()
    assert plan["a16"] == 1 and plan["BN"] > 192, plan
    if override:
        assert (plan["BN"], plan["splits"], plan["cluster"]) == override, plan
    ref = dict(inp, xq=xq, s_x=s_x)
    assert_close(y, O.layer_f64(ref), (spec, override))
    assert_close(y32, O.layer_f64(dict(ref, bias=np.zeros_like(inp["bias"]))), (spec, "f32"))
    _check_codes(ws, plan, xq)


@pytest.mark.parametrize("wl", ["conv64", "conv8_book16"])
def test_conv_f16_int8_form_equals_two_calls(wl):
    """The 64x64 W4A8 conv (both forms plan 192-wide tiles) and the 2^16-codebook 8x8 conv (the
    fused path) quantize to int8: the same bits as aq_quant_act + aq_conv2d_nhwc."""
    spec = WORKLOADS[wl]
    inp = make_conv(spec, seed=SEEDS[wl])
    x16, s_x, xq = _activations(spec, seed=3)
    y, ws, plan = _run(inp, x16, s_x)
    assert plan["a16"] == 0, plan
    _check_codes(ws, plan, xq)
    ref = dict(inp, xq=xq, s_x=s_x)
    y2 = run_conv(ref)
    assert np.array_equal(y, y2)
    assert_close(y, O.layer_f64(ref), wl)


def test_conv_f16_errors_and_empty():
    import torch
    import paper_2506_05960_gb300 as aq
    spec = ConvSpec(Nb=2, H=8, W=8, Cin=64, Cout=256, M=2)
    inp = make_conv(spec, seed=4)
    packed = pack(inp["codes"], 256, 9 * 64, 2, 8)
    x = dev(make_f16_activations((2, 8, 8, 64), seed=1))
    y = torch.empty((2, 8, 8, 256), dtype=torch.float16, device="cuda")
    shape = (2, 8, 8, 64, 256, 3, 3, 1, 1, 8, 2, 8)
    wsb = aq.aq_conv2d_f16_workspace_size(*shape, AUTO)
    assert wsb >= 2 * 2 * 8 * 8 * 64
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    books, scale = dev(inp["codebooks"]), dev(inp["scale"])
    with pytest.raises(aq.AQError) as e:                       # workspace too small
        aq.aq_conv2d_nhwc_f16(x, 0.02, packed, books, scale, None, y, aq.AQ_DTYPE_F16, *shape,
                              ws, 1024, AUTO)
    assert e.value.status == -5
    with pytest.raises(aq.AQError) as e:                       # s_x must be finite and > 0
        aq.aq_conv2d_nhwc_f16(x, 0.0, packed, books, scale, None, y, aq.AQ_DTYPE_F16, *shape,
                              ws, wsb, AUTO)
    assert e.value.status == -2
    with pytest.raises(aq.AQError) as e:                       # int8 output: the _q8 call
        aq.aq_conv2d_nhwc_f16(x, 0.02, packed, books, scale, None, y, aq.AQ_DTYPE_I8, *shape,
                              ws, wsb, AUTO)
    assert e.value.status == -3
    with pytest.raises(aq.AQError) as e:
        aq.aq_conv2d_nhwc_f16(None, 0.02, packed, books, scale, None, y, aq.AQ_DTYPE_F16, *shape,
                              ws, wsb, AUTO)
    assert e.value.status == -1
    aq.aq_conv2d_nhwc_f16(None, 0.02, None, None, None, None, None, aq.AQ_DTYPE_F16, 0,
                          *shape[1:], None, 0, AUTO)             # Nb == 0 is a no-op
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
