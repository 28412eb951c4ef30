"""GPU parity of the shared-memory A form of the tensor-core GEMM (aq_linear_a16, and
aq_linear_f16 on the dense paths): the 8-bit activations of Sec. 4.2.3 held as fp16 values,
both MMA operands read from shared memory, N tiles up to 256.

Checks: the same bits as aq_linear (int8 activations, TMEM A operand) when both run the
same plan (products of fp16 values are exact and the K order of the accumulation is the
same), and the layer tolerance against the fp64 oracle for every N tile, K split and
ragged shape."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_f16_activations, make_linear
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


def _layer(T, K, N, M=2, B=8, seed=0):
    inp = make_linear(LinearSpec(T=T, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5), seed=seed)
    packed = pack(inp["codes"], N, K, M, B)
    return inp, packed


def _run_a16(aq, inp, packed, out_f32, path=AUTO, with_bias=True, wdec=None):
    import torch
    T, K = inp["xq"].shape
    N, _, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    xh = dev(inp["xq"].astype(np.float16))
    wsb = aq.aq_linear_a16_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    if wdec is not None:
        ws[: wdec.numel() * 2].view(torch.float16).copy_(wdec.view(-1))
    y = poison((T, N), torch.float32 if out_f32 else torch.float16)
    aq.aq_linear_a16(xh, inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
                     dev(inp["bias"]) if with_bias else None, y,
                     aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, T, K, N, 8, M, B, ws, wsb,
                     path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.cpu().numpy()


def _run_i8(aq, inp, packed, out_f32, path=DENSE):
    import torch
    T, K = inp["xq"].shape
    N, _, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    wsb = aq.aq_linear_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    y = poison((T, N), torch.float32 if out_f32 else torch.float16)
    aq.aq_linear(dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
                 dev(inp["bias"]), y, aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, T, K, N, 8,
                 M, B, ws, wsb, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.cpu().numpy()


def _bits(y):
    return y.view(np.uint32 if y.dtype == np.float32 else np.uint16)


@pytest.mark.parametrize("T,K,N,M,B,out_f32", [
    (4096, 960, 2880, 2, 8, False),     # the qkv projection
    (300, 1024, 1152, 4, 8, True),      # ragged row tile, fp32 output
    (1000, 512, 264, 1, 16, False),     # 2^16 codebook, ragged N tile
    (200, 208, 208, 2, 8, True),        # ragged K block
])
def test_a16_equals_int8_form_same_plan(T, K, N, M, B, out_f32):
    import paper_2506_05960_gb300 as aq
    inp, packed = _layer(T, K, N, M, B, seed=T + K + N)
    pl = aq.aq_linear_plan(T, K, N, 8, M, B, DENSE)
    assert pl["a16"] == 0
    y8 = _run_i8(aq, inp, packed, out_f32)
    aq.aq_set_plan_override(pl["BN"], pl["splits"], pl["cluster"])
    try:
        pa = aq.aq_linear_a16_plan(T, K, N, 8, M, B, DENSE)
        assert (pa["BN"], pa["splits"], pa["cluster"], pa["a16"]) == (
            pl["BN"], pl["splits"], pl["cluster"], 1)
        ya = _run_a16(aq, inp, packed, out_f32, DENSE)
    finally:
        aq.aq_set_plan_override()
    assert np.array_equal(_bits(ya), _bits(y8))
    assert_close(ya.astype(np.float64), O.layer_f64(inp), (T, K, N, M, B))


@pytest.mark.parametrize("BN", [64, 96, 128, 160, 192, 224, 256])
@pytest.mark.parametrize("T,K,N", [(4096, 960, 2880), (300, 1024, 520)])
def test_a16_every_n_tile(BN, T, K, N):
    import paper_2506_05960_gb300 as aq
    inp, packed = _layer(T, K, N, seed=BN + T)
    aq.aq_set_plan_override(BN, 1, 0)
    try:
        pl = aq.aq_linear_a16_plan(T, K, N, 8, 2, 8, AUTO)
        assert pl["BN"] == BN and pl["splits"] == 1 and pl["a16"] == 1
        y = _run_a16(aq, inp, packed, False)
    finally:
        aq.aq_set_plan_override()
    assert_close(y.astype(np.float64), O.layer_f64(inp), (BN, T, K, N))


@pytest.mark.parametrize("BN,splits,cluster,out_f32", [
    (128, 4, 1, False),     # in-cluster split sum
    (256, 2, 1, True),      # the widest tile: its partial fills the ring
    (192, 3, 0, False),     # partials through the workspace + reduce kernel
    (64, 8, 1, True),
])
def test_a16_split_k(BN, splits, cluster, out_f32):
    import paper_2506_05960_gb300 as aq
    T, K, N = 256, 3072, 768
    inp, packed = _layer(T, K, N, seed=splits * 7 + BN)
    aq.aq_set_plan_override(BN, splits, cluster)
    try:
        pl = aq.aq_linear_a16_plan(T, K, N, 8, 2, 8, AUTO)
        assert (pl["BN"], pl["splits"], pl["cluster"]) == (BN, splits, cluster)
        y = _run_a16(aq, inp, packed, out_f32)
    finally:
        aq.aq_set_plan_override()
    assert_close(y.astype(np.float64), O.layer_f64(inp), (BN, splits, cluster))


def test_a16_predecoded_and_no_bias():
    import torch
    import paper_2506_05960_gb300 as aq
    T, K, N = 513, 960, 960
    inp, packed = _layer(T, K, N, seed=11)
    wdec = torch.empty((N, K), dtype=torch.float16, device="cuda")
    aq.aq_decode(packed, dev(inp["codebooks"]), wdec, N, K, 8, 2, 8)
    y_dense = _run_a16(aq, inp, packed, False, DENSE, with_bias=False)
    y_pre = _run_a16(aq, inp, packed, False, PRE, with_bias=False, wdec=wdec)
    assert np.array_equal(_bits(y_pre), _bits(y_dense))
    ref = O.layer_f64(dict(inp, bias=np.zeros_like(inp["bias"])))
    assert_close(y_dense.astype(np.float64), ref, "no bias")


def test_a16_tiny_and_ragged():
    import paper_2506_05960_gb300 as aq
    for (T, K, N) in ((1, 64, 64), (5, 80, 40), (129, 16, 8), (127, 1040, 392)):
        inp, packed = _layer(T, K, N, seed=T * 3 + N)
        y = _run_a16(aq, inp, packed, True)
        assert_close(y.astype(np.float64), O.layer_f64(inp), (T, K, N))


def test_a16_paths_and_errors():
    import torch
    import paper_2506_05960_gb300 as aq
    inp, packed = _layer(64, 256, 256, seed=5)
    for path in (FUSED, LUT, FEW):
        with pytest.raises(aq.AQError) as e:
            aq.aq_linear_a16_workspace_size(64, 256, 256, 8, 2, 8, path)
        assert e.value.status == -3
    wsb = aq.aq_linear_a16_workspace_size(64, 256, 256, 8, 2, 8, AUTO)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    xh = dev(inp["xq"].astype(np.float16))
    y = torch.empty((64, 256), dtype=torch.float16, device="cuda")
    args = (xh, inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]), None, y,
            aq.AQ_DTYPE_F16, 64, 256, 256, 8, 2, 8)
    with pytest.raises(aq.AQError) as e:                     # workspace too small
        aq.aq_linear_a16(*args, ws, wsb - 1024, AUTO)
    assert e.value.status == -5
    with pytest.raises(aq.AQError) as e:                     # int8 output: aq_linear_q8
        aq.aq_linear_a16(*args[:7], aq.AQ_DTYPE_I8, *args[8:], ws, wsb, AUTO)
    assert e.value.status == -3
    with pytest.raises(aq.AQError) as e:
        aq.aq_linear_a16(None, *args[1:], ws, wsb, AUTO)
    assert e.value.status == -1
    aq.aq_linear_a16(None, 0.02, None, None, None, None, None, aq.AQ_DTYPE_F16, 0, 256, 256, 8,
                     2, 8, None, 0, AUTO)                    # T == 0 is a no-op


def test_f16_quantizer_writes_codes_as_fp16():
    """aq_linear_f16 on the dense path keeps the quantized activations as fp16 values in
    its workspace: exactly the codes of aq_quant_act (the oracle's rule)."""
    import torch
    import paper_2506_05960_gb300 as aq
    T, K, N = 4096, 960, 2880
    inp, packed = _layer(T, K, N, seed=21)
    x16 = make_f16_activations((T, K), seed=4, std=2.0)
    s_x = float(np.float32(0.05))
    wsb = aq.aq_linear_f16_workspace_size(T, K, N, 8, 2, 8, AUTO)
    assert aq.aq_linear_f16_plan(T, K, N, 8, 2, 8, AUTO)["a16"] == 1
    ws = torch.full((wsb,), 0x55, dtype=torch.uint8, device="cuda")
    y = poison((T, N), torch.float16)
    aq.aq_linear_f16(dev(x16), s_x, packed, dev(inp["codebooks"]), dev(inp["scale"]),
                     dev(inp["bias"]), y, aq.AQ_DTYPE_F16, T, K, N, 8, 2, 8, ws, wsb, AUTO)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    codes = ws[: 2 * T * K].view(torch.float16).reshape(T, K).cpu().numpy()
    xq = O.quant_act(x16, s_x)
    assert np.array_equal(codes, xq.astype(np.float16))
    assert_close(y.cpu().numpy().astype(np.float64), O.layer_f64(dict(inp, xq=xq, s_x=s_x)), "f16")


@pytest.mark.parametrize("BN", [64, 128, 192, 256])
def test_a16_short_k_and_code_outputs(BN):
    """Tiles of at most 8 K blocks, and the next layer's codes as output, run the shared-memory
    A form with three epilogue warps per TMEM lane quarter (with N tile 64 one of the three has
    no chunk).  fp16 output against the oracle; the int8 codes and the fp16 codes equal the
    activation rule applied to the fp16 output, bit for bit."""
    import torch
    import paper_2506_05960_gb300 as aq
    T, K, N = 700, 384, 976          # ragged row tile; a ragged N tile for every BN
    inp, packed = _layer(T, K, N, seed=BN + 11)
    s_out = 0.05
    F16C, I8 = aq.AQ_DTYPE_F16_CODES, aq.AQ_DTYPE_I8
    xh = dev(inp["xq"].astype(np.float16))
    outs = {}
    aq.aq_set_plan_override(BN, 1, 0)
    try:
        pl = aq.aq_linear_a16_plan(T, K, N, 8, 2, 8, AUTO)
        assert pl["BN"] == BN and pl["a16"] == 1 and pl["splits"] == 1
        y = _run_a16(aq, inp, packed, False)
        for od in (I8, F16C):
            wsb = aq.aq_linear_ex_workspace_size(F16C, T, K, N, 8, 2, 8, AUTO)
            ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
            yo = (torch.full((T, N), 99, dtype=torch.int8, device="cuda") if od == I8
                  else poison((T, N), torch.float16))
            aq.aq_linear_ex(xh, F16C, inp["s_x"], packed, dev(inp["codebooks"]),
                            dev(inp["scale"]), dev(inp["bias"]), yo, od, s_out, T, K, N, 8, 2, 8,
                            ws, wsb, AUTO)
            torch.cuda.synchronize()
            assert aq.aq_device_error() == 0
            outs[od] = yo.cpu().numpy()
    finally:
        aq.aq_set_plan_override()
    assert_close(y.astype(np.float64), O.layer_f64(inp), (BN, T, K, N))
    q = O.quant_act(y, s_out)
    assert np.array_equal(outs[I8], q)
    assert np.array_equal(outs[F16C], q.astype(np.float16))
