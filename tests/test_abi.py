"""The C-ABI library builds, loads and exports every symbol of include/aq.h,
and its host-side validation rejects bad arguments without touching a GPU."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2506_05960_gb300 import _binding
    if not os.path.exists(_binding.library_path()):
        from paper_2506_05960_gb300.build import build
        build()
    return _binding.load_library()


def _declared_functions():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            names += re.findall(r"^AQ_API\s+[\w\s\*]+?\b(aq_\w+)\s*\(", text, flags=re.M)
    return names


def test_exports_every_declared_symbol(lib):
    names = _declared_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(lib, n), n
    assert lib.aq_abi_version() == 1


def test_binding_covers_header():
    from paper_2506_05960_gb300 import _binding
    assert set(_declared_functions()) == set(_binding._SIGNATURES)


def _declared_arity():
    """{name: parameter count} parsed from the AQ_API declarations."""
    out = {}
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            for m in re.finditer(r"^AQ_API\s+[\w\s\*]+?\b(aq_\w+)\s*\(([^)]*)\)", text,
                                 flags=re.M):
                params = m.group(2).strip()
                out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_arity_matches_header():
    from paper_2506_05960_gb300 import _binding
    arity = _declared_arity()
    for name, (_, args) in _binding._SIGNATURES.items():
        assert len(args) == arity[name], (name, len(args), arity[name])


def _size(fn, *args):
    out = ctypes.c_size_t(0)
    return fn(*args, ctypes.byref(out)), out.value


def test_packed_size(lib):
    r, v = _size(lib.aq_packed_size, 2880, 960, 8, 2, 8)
    assert r == 0 and v == 15 * 2880 * 16
    r, v = _size(lib.aq_packed_size, 960, 8640, 8, 1, 16)
    assert r == 0 and v == 135 * 960 * 16
    r, v = _size(lib.aq_packed_size, 8, 200, 8, 3, 8)          # ragged K: 4 blocks
    assert r == 0 and v == 4 * 8 * 8 * 3


@pytest.mark.parametrize("g,M,B,code", [(10, 2, 8, -3), (4, 2, 8, -3), (8, 0, 8, -3), (8, 9, 8, -3),
                                        (8, 3, 16, -3), (8, 2, 4, -3)])
def test_unsupported_formats(lib, g, M, B, code):
    r, _ = _size(lib.aq_packed_size, 64, 64, g, M, B)
    assert r == code
    assert b"unsupported" in lib.aq_last_error_string()


def test_shape_errors(lib):
    assert _size(lib.aq_packed_size, 64, 60, 8, 2, 8)[0] == -2          # K % g
    assert _size(lib.aq_linear_workspace_size, 4, 24, 64, 8, 2, 8, 0)[0] == -2   # K % 16
    assert _size(lib.aq_linear_workspace_size, 4, 64, 60, 8, 2, 8, 0)[0] == -2   # N % 8
    assert _size(lib.aq_linear_workspace_size, -1, 64, 64, 8, 2, 8, 0)[0] == -2
    # conv: Cin % 64, kernel size, stride
    assert _size(lib.aq_conv2d_workspace_size, 1, 8, 8, 48, 64, 3, 3, 1, 1, 8, 2, 8, 0)[0] == -3
    assert _size(lib.aq_conv2d_workspace_size, 1, 8, 8, 64, 64, 5, 5, 1, 2, 8, 2, 8, 0)[0] == -3
    assert _size(lib.aq_conv2d_workspace_size, 1, 8, 8, 64, 64, 3, 3, 3, 1, 8, 2, 8, 0)[0] == -3


def test_null_and_alignment_errors_do_not_launch(lib):
    # T > 0 with NULL pointers -> AQ_ERR_NULL before any CUDA call
    r = lib.aq_linear(None, 0.02, None, None, None, None, None, 0, 4, 64, 64, 8, 2, 8, None,
                      0, 0, None)
    assert r == -1
    # misaligned pointers (never dereferenced: validation fails first)
    r = lib.aq_linear(8 + 1, 0.02, 16, 16, 16, None, 16, 0, 4, 64, 64, 8, 2, 8, 16, 1 << 20,
                      0, None)
    assert r == -4
    # workspace too small (dense path: the decoded weights need N*K*2 bytes)
    r = lib.aq_linear(16, 0.02, 16, 16, 16, None, 16, 0, 256, 64, 64, 8, 2, 8, 16, 8, 1, None)
    assert r == -5
    # T == 0 is a no-op even with NULL buffers
    assert lib.aq_linear(None, 0.02, None, None, None, None, None, 0, 0, 64, 64, 8, 2, 8, None,
                         0, 0, None) == 0
    # ... and so are an empty batch of images and the fp16-input / int8-output variants
    assert lib.aq_conv2d_nhwc(None, 0.02, None, None, None, None, None, 0, 0, 8, 8, 64, 64, 3, 3,
                              1, 1, 8, 2, 8, None, 0, 0, None) == 0
    assert lib.aq_linear_f16(None, 0.02, None, None, None, None, None, 0, 0, 64, 64, 8, 2, 8,
                             None, 0, 0, None) == 0
    assert lib.aq_linear_q8(None, 0.02, None, None, None, None, None, 0.02, 0, 64, 64, 8, 2, 8,
                            None, 0, 0, None) == 0
    # quantizer: numel 0 no-op; bad scale
    assert lib.aq_quant_act(None, None, 0, 0.5, None) == 0
    assert lib.aq_quant_act(16, 16, 16, 0.0, None) == -2
    assert lib.aq_quant_act(16, 16, 16, float("nan"), None) == -2
    assert lib.aq_quant_act(16, 16, 16, float("inf"), None) == -2


def test_workspace_sizes(lib):
    r, v = _size(lib.aq_linear_workspace_size, 4096, 960, 2880, 8, 2, 8, 0)
    assert r == 0 and v >= 2880 * 960 * 2
    r, v = _size(lib.aq_conv2d_workspace_size, 16, 64, 64, 192, 192, 3, 3, 1, 1, 8, 4, 8, 0)
    assert r == 0 and v >= 192 * 1728 * 2


def test_kernel_aware_grouping_g9(lib):
    """g = 9 (one group per 3x3 filter): canonical layout stored as is, conv only,
    dense path only."""
    r, v = _size(lib.aq_packed_size, 96, 9 * 64, 9, 2, 8)
    assert r == 0 and v == 96 * 64 * 2
    r, v = _size(lib.aq_packed_size, 96, 9 * 64, 9, 1, 16)
    assert r == 0 and v == 96 * 64 * 2
    assert _size(lib.aq_packed_size, 96, 9 * 64 + 1, 9, 2, 8)[0] == -2          # K % 9
    # not a linear-layer format
    assert _size(lib.aq_linear_workspace_size, 128, 576, 64, 9, 2, 8, 0)[0] == -3
    # conv: AUTO and DENSE run the dense path, FUSED and LUT are refused
    for path in (0, 1):
        r, v = _size(lib.aq_conv2d_workspace_size, 2, 16, 16, 64, 96, 3, 3, 1, 1, 9, 2, 8, path)
        assert r == 0 and v >= 96 * 9 * 64 * 2
    for path in (2, 3):
        assert _size(lib.aq_conv2d_workspace_size, 2, 16, 16, 64, 96, 3, 3, 1, 1, 9, 2, 8,
                     path)[0] == -3



def test_plan_query_and_override(lib):
    """Plan introspection and the diagnostic plan override (no device access)."""
    import paper_2506_05960_gb300 as aq
    try:
        p = aq.aq_linear_plan(128, 960, 960)
        # one row tile: fused path, K split over a cluster, nothing in the workspace
        assert p["path"] == 2 and p["cluster"] == 1 and 2 <= p["splits"] <= 8
        assert aq.aq_linear_workspace_size(128, 960, 960) == 0
        assert aq.aq_linear_plan(4, 960, 960)["path"] == 4          # few tokens
        aq.aq_set_plan_override(64, 5, 0)
        p = aq.aq_linear_plan(128, 960, 960)
        assert (p["BN"], p["splits"], p["cluster"]) == (64, 5, 0)
        assert aq.aq_linear_workspace_size(128, 960, 960) == 5 * 128 * 960 * 4
        aq.aq_set_plan_override(0, 7, -1)                 # 15 K blocks cannot split 7 ways
        forced = aq.aq_linear_plan(128, 960, 960)
        aq.aq_set_plan_override()
        assert forced == aq.aq_linear_plan(128, 960, 960)  # the cost-model plan runs
        for bad in [(48, 0, -1), (-32, 0, -1), (256 + 32, 0, -1), (0, -1, -1), (0, 0, 2)]:
            with pytest.raises(aq.AQError) as e:
                aq.aq_set_plan_override(*bad)
            assert e.value.status == -2
        p = aq.aq_conv2d_plan(2, 8, 8, 960, 960, M=2)
        assert p["cluster"] == 1 and aq.aq_conv2d_workspace_size(2, 8, 8, 960, 960, M=2) == 0
        # fp16 activations on the dense paths: the shared-memory A form, N tiles up to 256;
        # int8 activations keep the TMEM A form (N tiles up to 192)
        assert aq.aq_linear_plan(4096, 960, 2880)["a16"] == 0
        pf = aq.aq_linear_f16_plan(4096, 960, 2880)
        assert pf["path"] == 1 and pf["a16"] == 1 and pf["stage_blocks"] >= 1
        assert aq.aq_linear_a16_plan(4096, 960, 2880) == pf
        assert aq.aq_linear_f16_plan(128, 960, 960)["a16"] == 0      # fused path: int8
        aq.aq_set_plan_override(256, 1, 0)
        assert aq.aq_linear_a16_plan(4096, 960, 2880)["BN"] == 256
        assert aq.aq_linear_plan(4096, 960, 2880)["BN"] <= 192       # falls back to the model
        aq.aq_set_plan_override()
        # the quantized activations are kept as fp16 values: 2*T*K bytes of workspace
        assert (aq.aq_linear_f16_workspace_size(4096, 960, 2880)
                >= 2 * 4096 * 960 + aq.aq_linear_a16_workspace_size(4096, 960, 2880))
        for path in (2, 3, 4):
            with pytest.raises(aq.AQError) as e:
                aq.aq_linear_a16_plan(64, 256, 256, path=path)
            assert e.value.status == -3
    finally:
        aq.aq_set_plan_override()


def test_missing_library_fails_loudly():
    """Without the compiled library every entry point raises: there is no Python or CPU
    fallback for any step of the path."""
    import subprocess
    import sys
    code = (
        "import paper_2506_05960_gb300._binding as b\n"
        "b._LIB_PATH = '/nonexistent/libaq_gb300.so'\n"
        "import paper_2506_05960_gb300 as aq\n"
        "try:\n"
        "    aq.aq_packed_size(256, 256, 8, 2, 8)\n"
        "except ImportError as e:\n"
        "    print('raised:', e)\n"
        "else:\n"
        "    print('no error')\n")
    r = subprocess.run([sys.executable, "-c", code], cwd=ROOT, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.startswith("raised:") and "no CPU fallback" in r.stdout, r.stdout


def test_plans_of_every_unet_layer_are_well_formed(lib):
    """Every layer shape of the UNet sweep, at batch 2, 16 and 64, both weight formats and
    every tensor-core path: the planner returns a runnable plan (host only, no device)."""
    import paper_2506_05960_gb300 as aq
    from aq_synth import unet_sweep_layers
    aq.aq_set_plan_override()
    n_checked = 0
    for batch in (2, 16, 64):
        for M in (2, 4):
            for kind, res, cin, cout, stride, _ in unet_sweep_layers():
                for path in (aq.AQ_PATH_AUTO, aq.AQ_PATH_DENSE, aq.AQ_PATH_FUSED,
                             aq.AQ_PATH_PREDECODED):
                    if kind == "conv3":
                        H = res * stride
                        T = batch * res * res
                        K = 9 * cin
                        p = aq.aq_conv2d_plan(batch, H, H, cin, cout, 3, 3, stride, 1, 8, M, 8,
                                              path)
                        ws = aq.aq_conv2d_workspace_size(batch, H, H, cin, cout, 3, 3, stride,
                                                         1, 8, M, 8, path)
                    else:
                        T, K = batch * res * res, cin
                        p = aq.aq_linear_plan(T, K, cout, 8, M, 8, path)
                        ws = aq.aq_linear_workspace_size(T, K, cout, 8, M, 8, path)
                    if p["path"] == aq.AQ_PATH_FEW_TOKENS:
                        assert ws == 0
                        continue
                    assert p["path"] in (aq.AQ_PATH_DENSE, aq.AQ_PATH_FUSED,
                                         aq.AQ_PATH_PREDECODED)
                    if path != aq.AQ_PATH_AUTO:
                        assert p["path"] == path
                    BN, S = p["BN"], p["splits"]
                    assert BN % 32 == 0 and 32 <= BN <= 192, p
                    assert p["stages"] >= 2, p
                    m_tiles = (T + 127) // 128
                    n_tiles = (cout + BN - 1) // BN
                    assert p["work_items"] == m_tiles * n_tiles * S, (p, T, cout)
                    k_blocks = (K + 63) // 64
                    assert 1 <= S <= k_blocks, p
                    if p["cluster"]:
                        assert 2 <= S <= 8, p
                    if p["path"] != aq.AQ_PATH_FUSED:
                        # the decoded weights (fp16, N x K) sit at the start of the workspace
                        assert ws >= cout * K * 2, (p, ws)
                    if S > 1 and not p["cluster"]:
                        assert ws >= S * T * cout * 4, (p, ws)   # fp32 split-K partials
                    n_checked += 1
    assert n_checked > 1000


def test_noalloc_argument_checks_before_any_cuda_call(lib):
    """aq_linear_noalloc refuses layers whose decoded weights exceed its fixed scratch
    (16 MiB) and bad arguments on the host, so these calls need no GPU."""
    args = lambda T, K, N, out=0, s=0.02: (None, s, None, None, None, None, None, out, T, K, N,
                                           8, 2, 8, None)
    assert lib.aq_linear_noalloc(*args(4, 4096, 2056)) == -5        # 4096*2056*2 > 16 MiB
    assert lib.aq_linear_noalloc(*args(4, 4096, 2048)) == -1        # fits: then NULL buffers
    assert lib.aq_linear_noalloc(*args(0, 4096, 2048)) == 0         # empty: no-op
    assert lib.aq_linear_noalloc(*args(4, 4096, 2048, out=2)) == -3  # int8 output not offered
    assert lib.aq_linear_noalloc(*args(4, 4096, 2048, s=float("nan"))) == -2
    assert lib.aq_linear_noalloc(*args(4, 4100, 2048)) == -2        # K % 16


def test_auto_path_rules(lib):
    """AUTO's choices for a linear layer (no device access): up to four tokens on a layer with
    at least 6 MB of 8-bit codes take the table path (one token with any M, more with 1, 2 or 4
    codebooks); few tokens otherwise the few-token kernel; one row tile the fused decode; more the dense path.  fp16 activations choose the
    shared-memory A form only where its plan has no K split and a wider N tile."""
    import paper_2506_05960_gb300 as aq
    LUT, FEW, FUSED, DENSE = 3, 4, 2, 1
    assert aq.aq_linear_plan(1, 8192, 16384, 8, 2, 8)["path"] == LUT       # 33.6 MB of codes
    assert aq.aq_linear_plan(1, 8192, 16384, 8, 1, 8)["path"] == LUT       # 16.8 MB
    assert aq.aq_linear_plan(1, 4096, 8192, 8, 2, 8)["path"] == LUT        # 8.4 MB
    assert aq.aq_linear_plan(1, 2048, 8192, 8, 2, 8)["path"] == FEW        # 4.2 MB
    assert aq.aq_linear_plan(1, 8192, 16384, 8, 1, 16)["path"] == FEW      # 16-bit codes
    assert aq.aq_linear_plan(2, 8192, 16384, 8, 2, 8)["path"] == LUT       # two tokens
    assert aq.aq_linear_plan(4, 8192, 16384, 8, 4, 8)["path"] == LUT       # four, 4x8
    assert aq.aq_linear_plan(4, 8192, 16384, 8, 3, 8)["path"] == FEW       # 3x8: general table
    assert aq.aq_linear_plan(5, 8192, 16384, 8, 2, 8)["path"] == FUSED     # five tokens
    assert aq.aq_linear_plan(1, 960, 2880, 8, 2, 8)["path"] == FEW
    assert aq.aq_linear_plan(100, 960, 2880, 8, 2, 8)["path"] == FUSED
    assert aq.aq_linear_plan(4096, 960, 2880, 8, 2, 8)["path"] == DENSE
    # the one-token table path needs a workspace for its per-chunk partial sums
    assert aq.aq_linear_workspace_size(1, 8192, 16384, 8, 2, 8) == \
        aq.aq_linear_workspace_size(1, 8192, 16384, 8, 2, 8, LUT) > 0
    for (T, K, N) in ((4096, 960, 2880), (16384, 192, 576), (2048, 960, 960)):
        p16, p8 = aq.aq_linear_f16_plan(T, K, N), aq.aq_linear_plan(T, K, N)
        wider = aq.aq_linear_a16_plan(T, K, N)
        want = wider["splits"] == 1 and wider["BN"] > p8["BN"]
        assert p16["a16"] == (1 if want else 0), (T, K, N, p16, p8, wider)


def _header_constants():
    """{name: int} of every AQ_* #define and enumerator with an integer value in include/*.h."""
    out = {}
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            for m in re.finditer(r"^#define\s+(AQ_\w+)\s+(-?\d+)\b", text, flags=re.M):
                out[m.group(1)] = int(m.group(2))
            for m in re.finditer(r"^\s*(AQ_(?:DTYPE|PATH)_\w+)\s*=\s*(-?\d+)", text, flags=re.M):
                out[m.group(1)] = int(m.group(2))
    return out


def test_binding_constants_match_header():
    """Status codes, dtype and path values, device error bits and the profile-kind count
    of the binding are the header's."""
    import paper_2506_05960_gb300 as aq
    from paper_2506_05960_gb300 import _binding
    c = _header_constants()
    dtypes = {k for k in c if k.startswith("AQ_DTYPE_")}
    paths = {k for k in c if k.startswith("AQ_PATH_")}
    deverrs = {k for k in c if k.startswith("AQ_DEVERR_")}
    errs = {k for k in c if k.startswith("AQ_ERR_")}
    assert len(dtypes) == 4 and len(paths) == 6 and len(deverrs) == 6 and len(errs) == 7
    for k in dtypes | paths | deverrs:
        assert getattr(aq, k) == c[k], k
    assert {v: k for k, v in _binding._ERRORS.items()} == {k: c[k] for k in errs}
    assert c["AQ_OK"] == 0 and len(aq.PROFILE_KINDS) == c["AQ_PROFILE_KINDS"]
    bits = sorted(c[k] for k in deverrs)
    assert bits == [1 << i for i in range(len(bits))]   # distinct single bits


def _lutr_fill(units, nrb, ctas, tau, build):
    """Greedy ranges: each CTA in turn takes as many chunk-major units as keep its row blocks
    plus `build` per chunk whose tables it builds within tau.  (placed all?, bounds)"""
    u, bounds = 0, [0]
    for _ in range(ctas):
        r = tau - build if u < units else 0
        while r > 0 and u < units:
            e = min(units, (u // nrb + 1) * nrb)
            if u + r <= e:
                u, r = u + r, 0
            else:
                r -= e - u + build
                u = e
        bounds.append(u)
    return u >= units, bounds


def _lutr_partition(units, nrb, ctas, build=64):
    lo, hi = build, units + build * (units // nrb + 2)
    while lo + 1 < hi:
        mid = (lo + hi) // 2
        if _lutr_fill(units, nrb, ctas, mid, build)[0]:
            hi = mid
        else:
            lo = mid
    return hi, _lutr_fill(units, nrb, ctas, hi, build)[1]


def _lutr_plan(T, K, N, M, sms=152, min_blocks=64):
    """The rotated-table kernel's chunks and CTA count: NT = 32 / TP code bytes per chunk;
    one CTA per SM with at least `min_blocks` (chunk, 32-row block) units each, or a whole
    multiple of the chunks when the balanced ranges' busiest CTA comes out cheaper."""
    tp = 1 if T == 1 else (2 if T == 2 else 4)
    nt = 32 // tp
    chunks = (((K + 63) // 64) * 8 * M + nt - 1) // nt
    nrb = (N + 31) // 32
    units = chunks * nrb
    ctas = max(1, min(sms, units // min_blocks))
    if chunks <= ctas:
        aligned = ctas // chunks * chunks
        if aligned < ctas and _lutr_partition(units, nrb, aligned)[0] < _lutr_partition(units, nrb, ctas)[0]:
            ctas = aligned
    return chunks, ctas


def test_table_ranges_cover_every_unit_once():
    """The balanced ranges are contiguous, ordered and cover all units; no CTA exceeds the
    bisected cost, and one unit less of budget cannot place them all."""
    for chunks, nrb, ctas in [(64, 512, 152), (64, 2048, 152), (32, 512, 128), (16, 17, 4),
                              (3, 1, 2), (1, 5000, 152)]:
        units = chunks * nrb
        tau, b = _lutr_partition(units, nrb, ctas)
        assert b[0] == 0 and b[-1] == units and len(b) == ctas + 1
        assert all(b[i] <= b[i + 1] for i in range(ctas))
        for i in range(ctas):
            if b[i + 1] > b[i]:
                touched = (b[i + 1] - 1) // nrb - b[i] // nrb + 1
                assert b[i + 1] - b[i] + 64 * touched <= tau
        assert not _lutr_fill(units, nrb, ctas, tau - 1, 64)[0]


@pytest.mark.parametrize("T,K,N,M,chunks,ctas", [
    (1, 8192, 16384, 2, 64, 152),
    (1, 8192, 65536, 2, 64, 152),
    (1, 4096, 8192, 2, 32, 128),     # aligned: every CTA inside one chunk is cheaper
    (2, 8192, 16384, 2, 128, 152),   # more chunks than SMs
    (1, 2048, 8192, 2, 16, 64),      # at least 64 row blocks per CTA
    (4, 1024, 528, 1, 16, 4),        # 272 units: 4 CTAs
])
def test_table_plan_chunks_and_ctas(lib, T, K, N, M, chunks, ctas):
    """The table path's plan query reports the rotated-table kernel's chunks and CTA count,
    and both follow the planning rule (restated here)."""
    import paper_2506_05960_gb300 as aq
    p = aq.aq_linear_plan(T, K, N, 8, M, 8, aq.AQ_PATH_LUT)
    assert p["path"] == aq.AQ_PATH_LUT
    assert (p["splits"], p["work_items"]) == (chunks, ctas) == _lutr_plan(T, K, N, M)


def test_table_plan_matches_rule_on_many_shapes(lib):
    import paper_2506_05960_gb300 as aq
    for T in (1, 2, 3, 4):
        for M in (1, 2, 4):
            for K in (512, 960, 2048, 4096, 8192):
                for N in (64, 1000, 2880, 16384):
                    p = aq.aq_linear_plan(T, K, N, 8, M, 8, aq.AQ_PATH_LUT)
                    assert (p["splits"], p["work_items"]) == _lutr_plan(T, K, N, M), (T, K, N, M)
