"""Failure detection of the tensor-core kernels without a GPU fault: every pipeline wait
is bounded, and a kernel whose wait runs out records an error bit, stops its other warps,
drains its own copies and MMAs, frees its tensor memory and returns.  The test shortens
the limit to 0 ns (aq_set_wait_limit_ns), so the first wait that is not already satisfied
gives up -- at the latest the epilogue's wait for the first accumulator, which needs a
whole tile's mainloop -- and checks that the call returns, that aq_device_error() reports
a time-out bit and nothing else, and that the next call with the default limit computes
the layer correctly on the same context."""

import numpy as np
import pytest

from aq_synth import LinearSpec, make_linear
from oracle import aq_oracle as O

from gpu_util import assert_close, dev, pack, poison

pytestmark = pytest.mark.gpu

AUTO, DENSE, FUSED = 0, 1, 2
TIMEOUT_BITS = 1 | 2 | 4 | 8 | 16


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()
    yield
    aq.aq_set_wait_limit_ns(-1)
    aq.aq_set_plan_override()


def _call(aq, inp, packed, path, form, limit_ns):
    """One layer call with the given wait limit; returns (y, device error word)."""
    import torch
    T, K = inp["xq"].shape
    N = inp["codes"].shape[0]
    if form == "a16":
        wsb = aq.aq_linear_a16_workspace_size(T, K, N, 8, 2, 8, path)
    else:
        wsb = aq.aq_linear_workspace_size(T, K, N, 8, 2, 8, path)
    ws = torch.empty(max(wsb, 16), dtype=torch.uint8, device="cuda")
    y = poison((T, N), torch.float16)
    args = (inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]), dev(inp["bias"]), y,
            aq.AQ_DTYPE_F16, T, K, N, 8, 2, 8, ws, wsb, path)
    aq.aq_set_wait_limit_ns(limit_ns)
    try:
        if form == "a16":
            aq.aq_linear_a16(dev(inp["xq"].astype(np.float16)), *args)
        else:
            aq.aq_linear(dev(inp["xq"]), *args)
    finally:
        aq.aq_set_wait_limit_ns(-1)
    torch.cuda.synchronize()          # the kernel returned on its own (no CUDA error)
    return y.cpu().numpy(), aq.aq_device_error()


@pytest.mark.parametrize("T,K,N,path,form,plan", [
    (4096, 960, 2880, DENSE, "i8", None),          # dense path, int8 activations (TMEM A)
    (4096, 960, 2880, DENSE, "a16", (256, 1, 0)),  # shared-memory A form, one CTA per tile
    (128, 960, 960, AUTO, "i8", None),             # fused decode, K split summed in a cluster
    (256, 3072, 768, DENSE, "a16", (128, 4, 1)),   # shared-memory A form, in-cluster split
])
def test_wait_timeout_reported_and_context_recovers(T, K, N, path, form, plan):
    import paper_2506_05960_gb300 as aq
    inp = make_linear(LinearSpec(T=T, K=K, N=N), seed=T + N + K)
    packed = pack(inp["codes"], N, K, 2, 8)
    assert aq.aq_device_error() == 0
    if plan:
        aq.aq_set_plan_override(*plan)
    try:
        if form == "i8" and path == AUTO:
            p = aq.aq_linear_plan(T, K, N, 8, 2, 8, path)
            assert p["path"] == FUSED and p["cluster"] == 1
        _, err = _call(aq, inp, packed, path, form, 0)
        assert err != 0 and (err & ~TIMEOUT_BITS) == 0, err
        # the default limit on the same context: a correct layer, no error
        y, err2 = _call(aq, inp, packed, path, form, -1)
    finally:
        aq.aq_set_plan_override()
    assert err2 == 0
    assert_close(y.astype(np.float64), O.layer_f64(inp), (T, K, N, path, form))
