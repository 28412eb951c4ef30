"""GPU parity of the codebook gradient (backward of Eq. 4, the continuous step of
Stage-2 fine-tuning, Sec. 3.2.1) against the fp64 oracle.  The kernel sums with
fp32 atomics in no fixed order, so each entry is compared within the fp32
accumulation bound: |dC - dC64| <= 1e-5 * (the same sum over |terms|)."""

import numpy as np
import pytest

from oracle import aq_oracle as O

from gpu_util import dev, pack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _run(codes, G, scale, s_x, N, K, g, M, B, calls=1):
    import torch
    import paper_2506_05960_gb300 as aq
    packed = pack(codes, N, K, M, B, g)
    dC = torch.zeros((M, 1 << B, g), dtype=torch.float32, device="cuda")
    for _ in range(calls):
        aq.aq_codebook_grad(packed, dev(G), dev(scale) if scale is not None else None, s_x, dC,
                            N, K, g, M, B)
    torch.cuda.synchronize()
    return dC.cpu().numpy().astype(np.float64)


def _check(dC, codes, Gf, scale, s_x, n_code, calls=1):
    ref = calls * O.codebook_grad_f64(codes, Gf, scale, s_x, n_code)
    bound = calls * O.codebook_grad_f64(codes, np.abs(Gf),
                                        None if scale is None else np.abs(scale), abs(s_x), n_code)
    assert np.all(np.abs(dC - ref) <= 1e-5 * bound + 1e-30)


@pytest.mark.parametrize("N,K,M,B", [(256, 256, 2, 8), (2880, 960, 2, 8), (96, 200, 3, 8),
                                     (64, 512, 8, 8), (960, 1024, 1, 16), (40, 264, 2, 16)])
def test_codebook_grad_g8(N, K, M, B):
    rng = np.random.default_rng(N + K + M)
    codes = rng.integers(0, 1 << B, size=(N, K // 8, M), dtype=np.uint8 if B == 8 else np.uint16)
    G = rng.normal(size=(N, K)).astype(np.float32)
    scale = rng.uniform(0.5, 1.5, size=N).astype(np.float16)
    dC = _run(codes, G, scale, 0.02, N, K, 8, M, B)
    _check(dC, codes, G, scale, 0.02, 1 << B)


@pytest.mark.parametrize("Cout,Cin,M,B", [(96, 64, 2, 8), (40, 37, 4, 8), (64, 128, 1, 16)])
def test_codebook_grad_kernel_aware(Cout, Cin, M, B):
    rng = np.random.default_rng(Cout + Cin)
    codes = rng.integers(0, 1 << B, size=(Cout, Cin, M), dtype=np.uint8 if B == 8 else np.uint16)
    G = rng.normal(size=(Cout, 9 * Cin)).astype(np.float32)        # OHWI columns
    dC = _run(codes, G, None, 0.5, Cout, 9 * Cin, 9, M, B)
    _check(dC, codes, O.kaq_from_ohwi(G.astype(np.float64)).reshape(Cout, -1), None, 0.5, 1 << B)


def test_codebook_grad_accumulates():
    rng = np.random.default_rng(7)
    N, K, M, B = 128, 256, 2, 8
    codes = rng.integers(0, 256, size=(N, K // 8, M), dtype=np.uint8)
    G = rng.normal(size=(N, K)).astype(np.float32)
    dC = _run(codes, G, None, 1.0, N, K, 8, M, B, calls=2)
    _check(dC, codes, G, None, 1.0, 256, calls=2)
