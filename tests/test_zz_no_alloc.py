"""aq_linear_noalloc: the linear layer for callers that cannot allocate device
memory (no workspace argument; the library's fixed 16 MiB scratch array holds
the decoded weights).

This file is named so that pytest collects it last: if it fails, a run that
stops at the first failure has already run every other test.  It passes alone
in a fresh process and after the other tests.
"""

import ctypes

import numpy as np
import pytest

from aq_synth import WORKLOADS, LinearSpec, make_linear
from oracle import aq_oracle as O


def test_noalloc_rejects_layers_beyond_the_scratch():
    """N*K*2 above the fixed scratch size fails with AQ_ERR_WORKSPACE before any CUDA call."""
    from paper_2506_05960_gb300 import _binding
    if not __import__("os").path.exists(_binding.library_path()):
        from paper_2506_05960_gb300.build import build
        build()
    lib = _binding.load_library()
    r = lib.aq_linear_noalloc(16, 0.02, 16, 16, 16, None, 16, 0, 4, 8192, 1032, 8, 2, 8, None)
    assert r == -5
    assert b"exceeds the fixed scratch" in lib.aq_last_error_string()


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row():
    import torch
    import paper_2506_05960_gb300 as aq
    from gpu_util import TOL_MAX_ABS, TOL_REL_FRO, dev, pack

    def layer_inputs(inp):
        T, K = inp["xq"].shape
        N, G, M = inp["codes"].shape
        B = 8 if inp["codes"].dtype == np.uint8 else 16
        return dict(T=T, K=K, N=N, M=M, B=B, xq=dev(inp["xq"]),
                    packed=pack(inp["codes"], N, K, M, B), books=dev(inp["codebooks"]),
                    scale=dev(inp["scale"]), bias=dev(inp["bias"]), s_x=inp["s_x"])

    def with_workspace(L):
        # aq_linear on the same path as the no-alloc call: decoded weights, no K split (any N
        # tile: each output's products are accumulated in the same K order)
        aq.aq_set_plan_override(0, 1, 0)
        try:
            ws_bytes = aq.aq_linear_workspace_size(L["T"], L["K"], L["N"], 8, L["M"], L["B"],
                                                   aq.AQ_PATH_DENSE)
            ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
            y = torch.full((L["T"], L["N"]), float("nan"), dtype=torch.float16, device="cuda")
            aq.aq_linear(L["xq"], L["s_x"], L["packed"], L["books"], L["scale"], L["bias"], y,
                         aq.AQ_DTYPE_F16, L["T"], L["K"], L["N"], 8, L["M"], L["B"], ws, ws_bytes,
                         aq.AQ_PATH_DENSE)
        finally:
            aq.aq_set_plan_override()
        return y

    def no_alloc(L):
        y = torch.full((L["T"], L["N"]), float("nan"), dtype=torch.float16, device="cuda")
        aq.aq_linear_noalloc(L["xq"], L["s_x"], L["packed"], L["books"], L["scale"], L["bias"],
                             y, aq.AQ_DTYPE_F16, L["T"], L["K"], L["N"], 8, L["M"], L["B"])
        return y

    # two different layers, one call each, back to back: the second call must not see
    # anything left in the shared scratch by the first
    inps = [make_linear(WORKLOADS["qkv"], seed=101),
            make_linear(LinearSpec(T=300, K=1024, N=1152, M=4, B=8, cb_std=0.025), seed=102)]
    layers = [layer_inputs(i) for i in inps]
    got = [no_alloc(L) for L in layers]
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    for inp, L, y in zip(inps, layers, got):
        ref = with_workspace(L)
        torch.cuda.synchronize()
        assert torch.equal(y.view(torch.int16), ref.view(torch.int16))   # bit for bit
        yn = y.float().cpu().numpy().astype(np.float64)
        m64 = O.compare(yn, O.layer_f64(inp))
        assert m64["rel_fro"] <= TOL_REL_FRO and m64["max_abs"] <= TOL_MAX_ABS * m64["scale_ref"], m64
