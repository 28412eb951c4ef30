"""GPU parity of the in-cluster split-K reduction: the K splits of an output tile
run as one thread-block cluster and are summed through distributed shared memory
in split order.  That is the order of the workspace split-K path (partials in
global memory + the reduce kernel), so both give the same bits; both are checked
against the fp64 oracle, on linear and convolution layers, all output types,
every cluster size 2..8, ragged row and column tiles, and more than one wave of
clusters."""

import numpy as np
import pytest

from aq_synth import ConvSpec, LinearSpec, make_conv, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack

pytestmark = pytest.mark.gpu

AUTO, DENSE, FUSED = 0, 1, 2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()
    yield
    aq.aq_set_plan_override()


@pytest.fixture(autouse=True)
def _default_plan():
    import paper_2506_05960_gb300 as aq
    aq.aq_set_plan_override()
    yield
    aq.aq_set_plan_override()


def _linear(inp, path, out, override=None):
    """Run aq_linear (out = 'f16' | 'f32') or aq_linear_q8 ('q8', scale from the
    oracle) under a plan override; returns (output array, plan dict)."""
    import torch
    import paper_2506_05960_gb300 as aq
    xq = inp["xq"]
    T, K = xq.shape
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    if override is not None:
        aq.aq_set_plan_override(*override)
    plan = aq.aq_linear_plan(T, K, N, 8, M, B, path)
    packed = pack(inp["codes"], N, K, M, B)
    ws_bytes = aq.aq_linear_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    args = (dev(xq), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
            dev(inp["bias"]))
    aq.aq_profile_enable(True)
    if out == "q8":
        y = torch.full((T, N), 99, dtype=torch.int8, device="cuda")
        aq.aq_linear_q8(*args, y, inp["s_out"], T, K, N, 8, M, B, ws, ws_bytes, path)
    else:
        f32 = out == "f32"
        y = torch.full((T, N), float("nan"), dtype=torch.float32 if f32 else torch.float16,
                       device="cuda")
        aq.aq_linear(*args, y, aq.AQ_DTYPE_F32 if f32 else aq.AQ_DTYPE_F16, T, K, N, 8, M, B,
                     ws, ws_bytes, path)
    torch.cuda.synchronize()
    prof = aq.aq_profile_read()
    aq.aq_profile_enable(False)
    assert aq.aq_device_error() == 0
    if override is not None:
        aq.aq_set_plan_override()
    plan["reduce_launches"] = prof["splitk"][1]
    return y.cpu().numpy(), plan


def _both(inp, path, out, BN, splits):
    yc, pc = _linear(inp, path, out, (BN, splits, 1))
    yw, pw = _linear(inp, path, out, (BN, splits, 0))
    assert (pc["BN"], pc["splits"], pc["cluster"]) == (BN, splits, 1), pc
    assert (pw["BN"], pw["splits"], pw["cluster"]) == (BN, splits, 0), pw
    assert pc["reduce_launches"] == 0 and pw["reduce_launches"] == 1
    return yc, yw


@pytest.mark.parametrize("splits,num_kb", [(2, 15), (3, 15), (4, 15), (5, 15), (6, 18),
                                           (7, 14), (8, 15)])
@pytest.mark.parametrize("path", [DENSE, FUSED])
def test_cluster_sizes_bitwise_equal_workspace_split(splits, num_kb, path):
    inp = make_linear(LinearSpec(T=128, K=64 * num_kb, N=320, M=2, B=8), seed=10 * splits + path)
    yc, yw = _both(inp, path, "f16", 64, splits)
    assert np.array_equal(yc.view(np.uint16), yw.view(np.uint16))
    assert_close(yc.astype(np.float64), O.layer_f64(inp), (splits, path))


@pytest.mark.parametrize("out", ["f16", "f32", "q8"])
def test_cluster_outputs_ragged_tiles(out):
    # T = 100: one ragged row tile; N = 976 with BN = 64: a ragged last column tile
    inp = make_linear(LinearSpec(T=100, K=960, N=976, M=2, B=8), seed=31)
    y64 = O.layer_f64(inp)
    inp["s_out"] = float(np.float32(0.8 * np.abs(y64).max() / 127.0))
    yc, yw = _both(inp, FUSED, out, 64, 5)
    if out == "f32":
        assert np.array_equal(yc.view(np.uint32), yw.view(np.uint32))
    elif out == "f16":
        assert np.array_equal(yc.view(np.uint16), yw.view(np.uint16))
    else:
        assert np.array_equal(yc, yw)
    if out != "q8":
        assert_close(yc.astype(np.float64), y64, out)
    else:
        ref = O.quant_act(y64.astype(np.float16), inp["s_out"])
        assert np.abs(yc.astype(np.int32) - ref.astype(np.int32)).max() <= 1


def test_cluster_many_row_tiles_beyond_one_wave():
    # 24 row tiles x 5 column tiles x 4 splits = 480 CTAs: clusters run in several waves
    inp = make_linear(LinearSpec(T=3000, K=1024, N=320, M=2, B=8), seed=41)
    yc, yw = _both(inp, DENSE, "f16", 64, 4)
    assert np.array_equal(yc.view(np.uint16), yw.view(np.uint16))
    assert_close(yc.astype(np.float64), O.layer_f64(inp))


def test_cluster_16bit_codes_and_more_codebooks():
    for M, B, seed in [(1, 16, 51), (4, 8, 52), (8, 8, 53)]:
        inp = make_linear(LinearSpec(T=96, K=1024, N=192, M=M, B=B, cb_std=0.05 / M ** 0.5),
                          seed=seed)
        yc, yw = _both(inp, FUSED, "f16", 64, 4)
        assert np.array_equal(yc.view(np.uint16), yw.view(np.uint16)), (M, B)
        assert_close(yc.astype(np.float64), O.layer_f64(inp), (M, B))


def test_auto_takes_cluster_split_for_small_token_counts():
    import paper_2506_05960_gb300 as aq
    for T, K, N in [(128, 960, 960), (128, 960, 2880), (64, 8640, 960)]:
        plan = aq.aq_linear_plan(T, K, N, 8, 2, 8, AUTO)
        assert plan["cluster"] == 1 and 2 <= plan["splits"] <= 8, (T, K, N, plan)
        assert aq.aq_linear_workspace_size(T, K, N, 8, 2, 8, AUTO) == 0
        inp = make_linear(LinearSpec(T=T, K=K, N=N, M=2, B=8), seed=T + K + N)
        y, p = _linear(inp, AUTO, "f16")
        assert p["reduce_launches"] == 0
        assert_close(y.astype(np.float64), O.layer_f64(inp), (T, K, N))


def _conv(inp, path, override):
    import torch
    import paper_2506_05960_gb300 as aq
    s = inp["spec"]
    N, G, M = inp["codes"].shape
    K = 9 * s.Cin
    aq.aq_set_plan_override(*override)
    plan = aq.aq_conv2d_plan(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, s.pad, 8, M, 8, path)
    packed = pack(inp["codes"], N, K, M, 8)
    ws_bytes = aq.aq_conv2d_workspace_size(s.Nb, s.H, s.W, s.Cin, s.Cout, 3, 3, s.stride, s.pad,
                                           8, M, 8, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    y = torch.full((s.Nb, s.Ho, s.Wo, s.Cout), float("nan"), dtype=torch.float16, device="cuda")
    aq.aq_conv2d_nhwc(dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]),
                      dev(inp["scale"]), dev(inp["bias"]), y, aq.AQ_DTYPE_F16, s.Nb, s.H, s.W,
                      s.Cin, s.Cout, 3, 3, s.stride, s.pad, 8, M, 8, ws, ws_bytes, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    aq.aq_set_plan_override()
    return y.cpu().numpy(), plan


@pytest.mark.parametrize("Nb,H,Cin,Cout,stride,path", [
    (2, 8, 960, 960, 1, FUSED),      # the 8 x 8 level of the UNet at batch 2
    (2, 16, 576, 576, 1, DENSE),
    (1, 16, 192, 200, 2, DENSE),     # stride 2, ragged output channels
])
def test_cluster_conv(Nb, H, Cin, Cout, stride, path):
    inp = make_conv(ConvSpec(Nb=Nb, H=H, W=H, Cin=Cin, Cout=Cout, stride=stride, M=2, B=8),
                    seed=H + Cin + stride)
    yc, pc = _conv(inp, path, (64, 4, 1))
    yw, pw = _conv(inp, path, (64, 4, 0))
    assert pc["cluster"] == 1 and pw["cluster"] == 0 and pc["splits"] == 4
    assert np.array_equal(yc.view(np.uint16), yw.view(np.uint16))
    assert_close(yc.astype(np.float64), O.layer_f64(inp))
