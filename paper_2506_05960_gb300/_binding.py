"""ctypes marshalling for the C ABI of ``include/aq.h`` (no computation here).

Pointer arguments accept a ``torch.Tensor`` (its ``data_ptr()``), a plain
integer address, or ``None`` (NULL).  ``stream`` defaults to the current torch
CUDA stream.  Every function returns what the C function returns through its
out-parameter (if any) and raises :class:`AQError` on a negative status.
"""

from __future__ import annotations

import ctypes
import os

_PKG = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_PKG, "lib", "libaq_gb300.so")

AQ_DTYPE_F16, AQ_DTYPE_F32, AQ_DTYPE_I8, AQ_DTYPE_F16_CODES = 0, 1, 2, 3
AQ_PATH_AUTO, AQ_PATH_DENSE, AQ_PATH_FUSED, AQ_PATH_LUT, AQ_PATH_FEW_TOKENS = 0, 1, 2, 3, 4
AQ_PATH_PREDECODED = 5

_ERRORS = {
    -1: "AQ_ERR_NULL", -2: "AQ_ERR_SHAPE", -3: "AQ_ERR_UNSUPPORTED", -4: "AQ_ERR_ALIGN",
    -5: "AQ_ERR_WORKSPACE", -6: "AQ_ERR_CUDA", -7: "AQ_ERR_DEVICE_TIMEOUT",
}

_c_int, _c_float, _c_size_t, _c_int64, _c_void_p = (
    ctypes.c_int, ctypes.c_float, ctypes.c_size_t, ctypes.c_int64, ctypes.c_void_p)

# name -> (restype, argtypes); mirrors include/aq.h
_SIGNATURES = {
    "aq_abi_version": (_c_int, []),
    "aq_last_error_string": (ctypes.c_char_p, []),
    "aq_device_error": (_c_int, [ctypes.POINTER(_c_int)]),
    "aq_profile_enable": (_c_int, [_c_int]),
    "aq_profile_read": (_c_int, [ctypes.POINTER(ctypes.c_double), ctypes.POINTER(_c_int64),
                                 _c_int]),
    "aq_packed_size": (_c_int, [_c_int] * 5 + [ctypes.POINTER(_c_size_t)]),
    "aq_pack": (_c_int, [_c_void_p, _c_void_p] + [_c_int] * 5 + [_c_void_p]),
    "aq_decode": (_c_int, [_c_void_p] * 3 + [_c_int] * 5 + [_c_void_p]),
    "aq_quant_act": (_c_int, [_c_void_p, _c_void_p, _c_int64, _c_float, _c_void_p]),
    "aq_codebook_grad": (_c_int, [_c_void_p] * 3 + [_c_float, _c_void_p] + [_c_int] * 5
                         + [_c_void_p]),
    "aq_code_update": (_c_int, [_c_void_p] * 4 + [_c_int] * 7 + [_c_void_p]),
    "aq_linear_input_grad_workspace_size": (_c_int, [_c_int] * 6 + [ctypes.POINTER(_c_size_t)]),
    "aq_linear_input_grad": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 4 + [_c_int] * 7
                             + [_c_void_p, _c_size_t, _c_void_p]),
    "aq_linear_workspace_size": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_size_t)]),
    "aq_linear_plan": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_set_plan_override": (_c_int, [_c_int] * 3),
    "aq_set_wait_limit_ns": (_c_int, [_c_int64]),
    "aq_linear_f16_workspace_size": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_size_t)]),
    "aq_linear_a16_workspace_size": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_size_t)]),
    "aq_linear_f16_plan": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_linear_a16_plan": (_c_int, [_c_int] * 7 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_linear_a16": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 7
                      + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_linear": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 7
                  + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_linear_f16": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 7
                      + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_linear_noalloc": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 7
                          + [_c_void_p]),
    "aq_linear_q8": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_float] + [_c_int] * 6
                     + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_conv2d_workspace_size": (_c_int, [_c_int] * 13 + [ctypes.POINTER(_c_size_t)]),
    "aq_conv2d_plan": (_c_int, [_c_int] * 13 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_conv2d_nhwc": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 13
                       + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_conv2d_nhwc_q8": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_float]
                          + [_c_int] * 12 + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_linear_ex_workspace_size": (_c_int, [_c_int] * 8 + [ctypes.POINTER(_c_size_t)]),
    "aq_linear_ex_plan": (_c_int, [_c_int] * 8 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_linear_ex": (_c_int, [_c_void_p, _c_int, _c_float] + [_c_void_p] * 5 + [_c_int, _c_float]
                     + [_c_int] * 6 + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_conv2d_ex_workspace_size": (_c_int, [_c_int] * 14 + [ctypes.POINTER(_c_size_t)]),
    "aq_conv2d_ex_plan": (_c_int, [_c_int] * 14 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_conv2d_nhwc_ex": (_c_int, [_c_void_p, _c_int, _c_float] + [_c_void_p] * 5
                          + [_c_int, _c_float] + [_c_int] * 12
                          + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
    "aq_conv2d_f16_workspace_size": (_c_int, [_c_int] * 13 + [ctypes.POINTER(_c_size_t)]),
    "aq_conv2d_f16_plan": (_c_int, [_c_int] * 13 + [ctypes.POINTER(_c_int), _c_int]),
    "aq_conv2d_nhwc_f16": (_c_int, [_c_void_p, _c_float] + [_c_void_p] * 5 + [_c_int] * 13
                           + [_c_void_p, _c_size_t, _c_int, _c_void_p]),
}

_lib = None


class AQError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where}: {_ERRORS.get(status, status)} ({msg})")
        self.status = status


def library_path() -> str:
    return _LIB_PATH


def load_library():
    """Load the shared library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise ImportError(
            f"{_LIB_PATH} is missing: build it with `python -m paper_2506_05960_gb300.build` "
            "(there is no CPU fallback)")
    lib = ctypes.CDLL(_LIB_PATH)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)} as a device pointer")


def _stream(stream):
    if stream is None:
        import torch
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status: int, where: str) -> None:
    if status != 0:
        raise AQError(status, where, load_library().aq_last_error_string().decode())


# --------------------------------------------------------------------------- API
def aq_abi_version() -> int:
    return load_library().aq_abi_version()


def aq_last_error_string() -> str:
    return load_library().aq_last_error_string().decode()


def aq_device_error() -> int:
    code = _c_int(0)
    _check(load_library().aq_device_error(ctypes.byref(code)), "aq_device_error")
    return code.value


PROFILE_KINDS = ("quant", "pack", "decode", "gemm", "splitk", "lut_build", "lut_gather",
                 "fused_gemm")


def aq_profile_enable(on: bool = True) -> None:
    _check(load_library().aq_profile_enable(1 if on else 0), "aq_profile_enable")


def aq_profile_read() -> dict:
    """{kind: (milliseconds, launches)} since the last aq_profile_enable()."""
    n = len(PROFILE_KINDS)
    ms = (ctypes.c_double * n)()
    cnt = (_c_int64 * n)()
    _check(load_library().aq_profile_read(ms, cnt, n), "aq_profile_read")
    return {k: (ms[i], cnt[i]) for i, k in enumerate(PROFILE_KINDS)}


def aq_packed_size(N, K, g=8, M=2, B=8) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_packed_size(N, K, g, M, B, ctypes.byref(out)), "aq_packed_size")
    return out.value


def aq_pack(codes_canon, codes_packed, N, K, g=8, M=2, B=8, stream=None) -> None:
    _check(load_library().aq_pack(_ptr(codes_canon), _ptr(codes_packed), N, K, g, M, B,
                                  _stream(stream)), "aq_pack")


def aq_decode(codes_packed, codebooks, W_out, N, K, g=8, M=2, B=8, stream=None) -> None:
    _check(load_library().aq_decode(_ptr(codes_packed), _ptr(codebooks), _ptr(W_out), N, K, g,
                                    M, B, _stream(stream)), "aq_decode")


def aq_quant_act(x, xq, numel, s_x, stream=None) -> None:
    _check(load_library().aq_quant_act(_ptr(x), _ptr(xq), int(numel), float(s_x),
                                       _stream(stream)), "aq_quant_act")


def aq_codebook_grad(codes_packed, G, scale, s_x, dC, N, K, g=8, M=2, B=8, stream=None) -> None:
    """dC += the codebook gradient of the groups' codewords (dC accumulates)."""
    _check(load_library().aq_codebook_grad(
        _ptr(codes_packed), _ptr(G), _ptr(scale), float(s_x), _ptr(dC), N, K, g, M, B,
        _stream(stream)), "aq_codebook_grad")


def aq_linear_input_grad_workspace_size(T, K, N, g=8, M=2, B=8) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_linear_input_grad_workspace_size(T, K, N, g, M, B, ctypes.byref(out)),
           "aq_linear_input_grad_workspace_size")
    return out.value


def aq_linear_input_grad(dy, alpha, codes_packed, codebooks, scale, dx, out_dtype, T, K, N, g=8,
                         M=2, B=8, workspace=None, workspace_bytes=0, stream=None) -> None:
    """dX = alpha * dY diag(scale) W-hat (the layer's input gradient)."""
    _check(load_library().aq_linear_input_grad(
        _ptr(dy), float(alpha), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(dx),
        out_dtype, T, K, N, g, M, B, _ptr(workspace), int(workspace_bytes), _stream(stream)),
        "aq_linear_input_grad")


def aq_code_update(W, codebooks, codes, H, m_first, m_count, N, K, g=8, M=2, B=8,
                   stream=None) -> None:
    """One greedy code-search step over codebooks [m_first, m_first + m_count)."""
    _check(load_library().aq_code_update(
        _ptr(W), _ptr(codebooks), _ptr(codes), _ptr(H), m_first, m_count, N, K, g, M, B,
        _stream(stream)), "aq_code_update")


def aq_linear_workspace_size(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_linear_workspace_size(T, K, N, g, M, B, path, ctypes.byref(out)),
           "aq_linear_workspace_size")
    return out.value


_PLAN_KEYS = ("path", "BN", "splits", "cluster", "stages", "work_items", "a16", "stage_blocks")


def aq_set_plan_override(BN=0, splits=0, cluster=-1) -> None:
    """Restrict this thread's later tensor-core plans (diagnostics); no arguments: default."""
    _check(load_library().aq_set_plan_override(BN, splits, cluster), "aq_set_plan_override")


def _plan(fn, name, *args) -> dict:
    n = len(_PLAN_KEYS)
    info = (_c_int * n)()
    _check(fn(*args, info, n), name)
    return dict(zip(_PLAN_KEYS, list(info)))


AQ_DEVERR_TIMEOUT_FULL, AQ_DEVERR_TIMEOUT_EMPTY, AQ_DEVERR_TIMEOUT_CONV = 1, 2, 4
AQ_DEVERR_TIMEOUT_ACCUM, AQ_DEVERR_TIMEOUT_DRAIN, AQ_DEVERR_SMEM_LAYOUT = 8, 16, 32


def aq_set_wait_limit_ns(ns=-1) -> None:
    """Failure-path tests: later tensor-core launches of this thread give up a pipeline
    wait after ns nanoseconds (ns < 0: the default, about two seconds)."""
    _check(load_library().aq_set_wait_limit_ns(int(ns)), "aq_set_wait_limit_ns")


def aq_linear_plan(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> dict:
    """The plan aq_linear runs for these shapes (diagnostics; no device access)."""
    return _plan(load_library().aq_linear_plan, "aq_linear_plan", T, K, N, g, M, B, path)


def aq_linear_f16_plan(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> dict:
    """The plan aq_linear_f16 runs for these shapes (diagnostics; no device access)."""
    return _plan(load_library().aq_linear_f16_plan, "aq_linear_f16_plan", T, K, N, g, M, B, path)


def aq_linear_a16_plan(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> dict:
    """The plan aq_linear_a16 runs for these shapes (diagnostics; no device access)."""
    return _plan(load_library().aq_linear_a16_plan, "aq_linear_a16_plan", T, K, N, g, M, B, path)


def aq_linear(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, T, K, N, g=8, M=2,
              B=8, workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    _check(load_library().aq_linear(
        _ptr(xq), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, T, K, N, g, M, B, _ptr(workspace), int(workspace_bytes), path,
        _stream(stream)), "aq_linear")


def aq_linear_f16_workspace_size(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_linear_f16_workspace_size(T, K, N, g, M, B, path, ctypes.byref(out)),
           "aq_linear_f16_workspace_size")
    return out.value


def aq_linear_f16(x, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, T, K, N, g=8, M=2,
                  B=8, workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """aq_quant_act + aq_linear in one call from fp16 activations x (codes kept in workspace)."""
    _check(load_library().aq_linear_f16(
        _ptr(x), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, T, K, N, g, M, B, _ptr(workspace), int(workspace_bytes), path,
        _stream(stream)), "aq_linear_f16")


def aq_linear_a16_workspace_size(T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_linear_a16_workspace_size(T, K, N, g, M, B, path, ctypes.byref(out)),
           "aq_linear_a16_workspace_size")
    return out.value


def aq_linear_a16(xh, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, T, K, N, g=8, M=2,
                  B=8, workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """aq_linear on 8-bit activations held as fp16 values (dense paths)."""
    _check(load_library().aq_linear_a16(
        _ptr(xh), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, T, K, N, g, M, B, _ptr(workspace), int(workspace_bytes), path,
        _stream(stream)), "aq_linear_a16")


def aq_linear_q8(xq, s_x, codes_packed, codebooks, scale, bias, yq, s_out, T, K, N, g=8, M=2,
                 B=8, workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """aq_linear whose epilogue writes the next layer's int8 activations (scale s_out)."""
    _check(load_library().aq_linear_q8(
        _ptr(xq), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(yq), float(s_out), T, K, N, g, M, B, _ptr(workspace), int(workspace_bytes), path,
        _stream(stream)), "aq_linear_q8")


def aq_linear_noalloc(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, T, K, N,
                      g=8, M=2, B=8, stream=None) -> None:
    """aq_linear with the library's fixed device scratch instead of a caller workspace."""
    _check(load_library().aq_linear_noalloc(
        _ptr(xq), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, T, K, N, g, M, B, _stream(stream)), "aq_linear_noalloc")


def aq_conv2d_workspace_size(Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8,
                             path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_conv2d_workspace_size(Nb, H, W, Cin, Cout, kh, kw, stride, pad, g,
                                                   M, B, path, ctypes.byref(out)),
           "aq_conv2d_workspace_size")
    return out.value


def aq_conv2d_plan(Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8,
                   path=AQ_PATH_AUTO) -> dict:
    """The plan aq_conv2d_nhwc runs for these shapes (diagnostics; no device access)."""
    return _plan(load_library().aq_conv2d_plan, "aq_conv2d_plan", Nb, H, W, Cin, Cout, kh, kw,
                 stride, pad, g, M, B, path)


def aq_conv2d_nhwc(xq, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, Nb, H, W, Cin,
                   Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8, workspace=None,
                   workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    _check(load_library().aq_conv2d_nhwc(
        _ptr(xq), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, _ptr(workspace),
        int(workspace_bytes), path, _stream(stream)), "aq_conv2d_nhwc")


def aq_conv2d_nhwc_q8(xq, s_x, codes_packed, codebooks, scale, bias, yq, s_out, Nb, H, W, Cin,
                      Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8, workspace=None,
                      workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """aq_conv2d_nhwc whose epilogue writes the next layer's int8 activations (scale s_out)."""
    _check(load_library().aq_conv2d_nhwc_q8(
        _ptr(xq), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(yq), float(s_out), Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B,
        _ptr(workspace), int(workspace_bytes), path, _stream(stream)), "aq_conv2d_nhwc_q8")


def aq_conv2d_f16_workspace_size(Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4,
                                 B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_conv2d_f16_workspace_size(Nb, H, W, Cin, Cout, kh, kw, stride, pad,
                                                       g, M, B, path, ctypes.byref(out)),
           "aq_conv2d_f16_workspace_size")
    return out.value


def aq_conv2d_f16_plan(Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8,
                       path=AQ_PATH_AUTO) -> dict:
    """The plan aq_conv2d_nhwc_f16 runs for these shapes (diagnostics; no device access)."""
    return _plan(load_library().aq_conv2d_f16_plan, "aq_conv2d_f16_plan", Nb, H, W, Cin, Cout,
                 kh, kw, stride, pad, g, M, B, path)


def aq_conv2d_nhwc_f16(x, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, Nb, H, W, Cin,
                       Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8, workspace=None,
                       workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """aq_quant_act + aq_conv2d_nhwc in one call from fp16 NHWC activations."""
    _check(load_library().aq_conv2d_nhwc_f16(
        _ptr(x), float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale), _ptr(bias),
        _ptr(y), out_dtype, Nb, H, W, Cin, Cout, kh, kw, stride, pad, g, M, B, _ptr(workspace),
        int(workspace_bytes), path, _stream(stream)), "aq_conv2d_nhwc_f16")


def aq_linear_ex_workspace_size(act_dtype, T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_linear_ex_workspace_size(act_dtype, T, K, N, g, M, B, path,
                                                      ctypes.byref(out)),
           "aq_linear_ex_workspace_size")
    return out.value


def aq_linear_ex_plan(act_dtype, T, K, N, g=8, M=2, B=8, path=AQ_PATH_AUTO) -> dict:
    """The plan aq_linear_ex runs for these shapes and activation kind (no device access)."""
    return _plan(load_library().aq_linear_ex_plan, "aq_linear_ex_plan", act_dtype, T, K, N, g,
                 M, B, path)


def aq_linear_ex(act, act_dtype, s_x, codes_packed, codebooks, scale, bias, y, out_dtype, s_out,
                 T, K, N, g=8, M=2, B=8, workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO,
                 stream=None) -> None:
    """The linear layer with the activation kind (int8 or fp16 codes) and the output kind
    (fp16, fp32, int8 codes or fp16 codes with scale s_out) as arguments."""
    _check(load_library().aq_linear_ex(
        _ptr(act), act_dtype, float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale),
        _ptr(bias), _ptr(y), out_dtype, float(s_out), T, K, N, g, M, B, _ptr(workspace),
        int(workspace_bytes), path, _stream(stream)), "aq_linear_ex")


def aq_conv2d_ex_workspace_size(act_dtype, Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1,
                                g=8, M=4, B=8, path=AQ_PATH_AUTO) -> int:
    out = _c_size_t(0)
    _check(load_library().aq_conv2d_ex_workspace_size(act_dtype, Nb, H, W, Cin, Cout, kh, kw,
                                                      stride, pad, g, M, B, path,
                                                      ctypes.byref(out)),
           "aq_conv2d_ex_workspace_size")
    return out.value


def aq_conv2d_ex_plan(act_dtype, Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4,
                      B=8, path=AQ_PATH_AUTO) -> dict:
    """The plan aq_conv2d_nhwc_ex runs for these shapes and activation kind (no device access)."""
    return _plan(load_library().aq_conv2d_ex_plan, "aq_conv2d_ex_plan", act_dtype, Nb, H, W, Cin,
                 Cout, kh, kw, stride, pad, g, M, B, path)


def aq_conv2d_nhwc_ex(act, act_dtype, s_x, codes_packed, codebooks, scale, bias, y, out_dtype,
                      s_out, Nb, H, W, Cin, Cout, kh=3, kw=3, stride=1, pad=1, g=8, M=4, B=8,
                      workspace=None, workspace_bytes=0, path=AQ_PATH_AUTO, stream=None) -> None:
    """The 3x3 NHWC convolution with the activation and output kinds as arguments."""
    _check(load_library().aq_conv2d_nhwc_ex(
        _ptr(act), act_dtype, float(s_x), _ptr(codes_packed), _ptr(codebooks), _ptr(scale),
        _ptr(bias), _ptr(y), out_dtype, float(s_out), Nb, H, W, Cin, Cout, kh, kw, stride, pad,
        g, M, B, _ptr(workspace), int(workspace_bytes), path, _stream(stream)),
           "aq_conv2d_nhwc_ex")
