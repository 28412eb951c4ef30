"""GPU parity of the layer's input gradient (aq_linear_input_grad: dX = alpha * dY diag(scale)
W-hat, the backward pass through the AQ layer of the Sec. 3.2.1 continuous step): the
transposed, scaled decode bit for bit against its rule, and the result within the layer
tolerance of the fp64 oracle, through the same decode + tensor-core contraction as the
forward layer."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, poison

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _grad(inp, dy, alpha, out_f32=False):
    import torch
    import paper_2506_05960_gb300 as aq
    N, Gr, M = inp["codes"].shape
    K = Gr * 8
    T = dy.shape[0]
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    packed = pack(inp["codes"], N, K, M, B)
    wsb = aq.aq_linear_input_grad_workspace_size(T, K, N, 8, M, B)
    ws = torch.full((wsb,), 0x7F, dtype=torch.uint8, device="cuda")
    dx = poison((T, K), torch.float32 if out_f32 else torch.float16)
    aq.aq_linear_input_grad(dev(dy), alpha, packed, dev(inp["codebooks"]), dev(inp["scale"]), dx,
                            aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, T, K, N, 8, M, B,
                            ws, wsb)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return dx.float().cpu().numpy().astype(np.float64), ws


def _dy(T, N, seed):
    return np.random.default_rng(seed).normal(0, 1, size=(T, N)).astype(np.float16)


@pytest.mark.parametrize("T,K,N,M,B,alpha,out_f32", [
    (4096, 960, 2880, 2, 8, 1.0, False),     # the qkv projection, dL/dX
    (4096, 2880, 960, 2, 8, 0.02, True),     # its transpose shape, dL/dxq (alpha = s_x)
    (300, 208, 144, 1, 16, 1.0, True),       # 2^16 codebook, ragged M, K and N tiles
    (128, 256, 4096, 4, 8, 1.0, False),      # long reduction over N (split-K plans)
    (1, 64, 64, 2, 8, 0.5, False),           # one token
])
def test_input_grad_matches_oracle(T, K, N, M, B, alpha, out_f32):
    inp = make_linear(LinearSpec(T=8, K=K, N=N, M=M, B=B, cb_std=0.05 / M ** 0.5),
                      seed=K + N + M)
    dy = _dy(T, N, T + K)
    dx, ws = _grad(inp, dy, alpha, out_f32)
    ref = O.input_grad_f64(dy, inp["codes"], inp["codebooks"], inp["scale"], alpha)
    assert_close(dx, ref, (T, K, N, M, B, alpha))
    # the workspace starts with the transposed, scaled weight: fp16(scale[n] * W-hat[n][k]),
    # W-hat by the decode rule, the product of two fp16 values rounded once to fp16
    wt = ws[: K * N * 2].cpu().numpy().view(np.float16).reshape(K, N)
    rule = O.decode_rule_f16(inp["codes"], inp["codebooks"]).astype(np.float32)
    want = (rule * inp["scale"].astype(np.float32)[:, None]).astype(np.float16).T
    assert np.array_equal(wt.view(np.uint16), want.view(np.uint16))


def test_input_grad_errors_and_empty():
    import torch
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=8, K=256, N=256), seed=5)
    packed = pack(inp["codes"], 256, 256, 2, 8)
    dy = dev(_dy(16, 256, 1))
    dx = torch.empty((16, 256), dtype=torch.float16, device="cuda")
    wsb = aq.aq_linear_input_grad_workspace_size(16, 256, 256, 8, 2, 8)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    args = (dy, 1.0, packed, dev(inp["codebooks"]), dev(inp["scale"]), dx, aq.AQ_DTYPE_F16, 16,
            256, 256, 8, 2, 8)
    with pytest.raises(aq.AQError) as e:                       # workspace too small
        aq.aq_linear_input_grad(*args, ws, wsb - 1024)
    assert e.value.status == -5
    with pytest.raises(aq.AQError) as e:                       # N % 16
        aq.aq_linear_input_grad_workspace_size(16, 256, 248, 8, 2, 8)
    assert e.value.status == -2
    with pytest.raises(aq.AQError) as e:                       # alpha must be finite
        aq.aq_linear_input_grad(dy, float("inf"), *args[2:], ws, wsb)
    assert e.value.status == -2
    aq.aq_linear_input_grad(None, 1.0, None, None, None, None, aq.AQ_DTYPE_F16, 0, 256, 256, 8,
                            2, 8, None, 0)                      # T == 0 is a no-op
