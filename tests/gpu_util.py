"""Helpers for the GPU parity tests: move seeded inputs to the device and run
the library through its C ABI.  No arithmetic of the method lives here."""

import numpy as np

TOL_REL_FRO = 2e-3      # relative Frobenius error bound vs the fp64 oracle
TOL_MAX_ABS = 1e-2      # max |error| bound, as a fraction of max |y64|


def dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def poison(shape, dtype):
    import torch
    return torch.full(shape, float("nan"), dtype=dtype, device="cuda")


def pack(codes, N, K, M, B, g=8):
    import torch
    import paper_2506_05960_gb300 as aq
    packed = torch.empty(aq.aq_packed_size(N, K, g, M, B), dtype=torch.uint8, device="cuda")
    aq.aq_pack(dev(codes), packed, N, K, g, M, B)
    return packed


def run_linear(inp, out_f32=False, with_bias=True, path=0):
    import torch
    import paper_2506_05960_gb300 as aq
    xq = inp["xq"]
    T, K = xq.shape
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    packed = pack(inp["codes"], N, K, M, B)
    ws_bytes = aq.aq_linear_workspace_size(T, K, N, 8, M, B, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    y = poison((T, N), torch.float32 if out_f32 else torch.float16)
    aq.aq_linear(dev(xq), inp["s_x"], packed, dev(inp["codebooks"]), dev(inp["scale"]),
                 dev(inp["bias"]) if with_bias else None, y,
                 aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, T, K, N, 8, M, B, ws, ws_bytes,
                 path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.float().cpu().numpy().astype(np.float64)


def run_conv(inp, out_f32=False, with_bias=True, path=0):
    import torch
    import paper_2506_05960_gb300 as aq
    s = inp["spec"]
    N, G, M = inp["codes"].shape
    B = 8 if inp["codes"].dtype == np.uint8 else 16
    K = s.kh * s.kw * s.Cin
    g = s.g                               # 8, or 9 for one group per 3x3 filter
    packed = pack(inp["codes"], N, K, M, B, g)
    ws_bytes = aq.aq_conv2d_workspace_size(s.Nb, s.H, s.W, s.Cin, s.Cout, s.kh, s.kw, s.stride,
                                           s.pad, g, M, B, path)
    ws = torch.empty(max(ws_bytes, 16), dtype=torch.uint8, device="cuda")
    y = poison((s.Nb, s.Ho, s.Wo, s.Cout), torch.float32 if out_f32 else torch.float16)
    aq.aq_conv2d_nhwc(dev(inp["xq"]), inp["s_x"], packed, dev(inp["codebooks"]),
                      dev(inp["scale"]), dev(inp["bias"]) if with_bias else None, y,
                      aq.AQ_DTYPE_F32 if out_f32 else aq.AQ_DTYPE_F16, s.Nb, s.H, s.W, s.Cin,
                      s.Cout, s.kh, s.kw, s.stride, s.pad, g, M, B, ws, ws_bytes, path)
    torch.cuda.synchronize()
    assert aq.aq_device_error() == 0
    return y.float().cpu().numpy().astype(np.float64)


def assert_close(y, y64, what=""):
    from oracle import aq_oracle as O
    m = O.compare(y, y64)
    assert m["rel_fro"] <= TOL_REL_FRO, (what, m)
    assert m["max_abs"] <= TOL_MAX_ABS * m["scale_ref"], (what, m)
    return m
