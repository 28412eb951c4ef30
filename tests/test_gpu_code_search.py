"""GPU parity of the greedy code-search step (Stage-1 calibration, Sec. 3.1):
bit-exact codes against the reference step (same fp32 decision rule), with and
without the calibration-input weighting, on one codebook and on a sweep over all;
and, independently of that rule's operation order, every chosen code is a float64
minimiser of its group's error up to float32 near-ties."""

import numpy as np
import pytest

from oracle import aq_oracle as O

from gpu_util import dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


def _step(W, books, codes, H, m_first, m_count):
    import torch
    import paper_2506_05960_gb300 as aq
    N, Gr, M = codes.shape
    c = dev(codes)
    aq.aq_code_update(dev(W), dev(books), c, dev(H) if H is not None else None, m_first, m_count,
                      N, Gr * 8, 8, M, 8)
    torch.cuda.synchronize()
    return c.cpu().numpy()


@pytest.mark.parametrize("N,Gr,M,weighted,m_first,m_count", [
    (64, 12, 2, False, 0, 2),
    (37, 5, 3, True, 1, 2),
    (256, 16, 1, False, 0, 1),
    (48, 8, 4, True, 0, 4),
])
def test_code_update_bit_exact(N, Gr, M, weighted, m_first, m_count):
    rng = np.random.default_rng(N + Gr + M)
    books = rng.normal(0, 0.05, size=(M, 256, 8)).astype(np.float16)
    W = rng.normal(0, 0.05 * M ** 0.5, size=(N, Gr * 8)).astype(np.float32)
    codes = rng.integers(0, 256, size=(N, Gr, M), dtype=np.uint8)
    H = None
    if weighted:
        A = rng.normal(size=(Gr, 8, 32)).astype(np.float32)
        H = np.einsum("iek,ifk->ief", A, A).astype(np.float32)
    got = _step(W, books, codes, H, m_first, m_count)
    ref = O.code_update_f32(W, books, codes, H, ms=range(m_first, m_first + m_count))
    assert np.array_equal(got, ref)
    _assert_near_minimisers(W, books, codes, got, H, m_first, m_count)


def _assert_near_minimisers(W, books, old, new, H, m_first, m_count):
    """Independent of the reference step's operation order: each code the GPU chose for
    codebook m is, in float64, a minimiser of its group's error over all 256 codewords --
    with the codebooks updated before m at their new codes and those after m at their old
    ones -- up to float32 near-ties."""
    N, Gr, M = old.shape
    C = books.astype(np.float64)                                    # [M][256][8]
    Wg = W.astype(np.float64).reshape(N, Gr, 8)
    for m in range(m_first, m_first + m_count):
        ctx = np.where(np.arange(M)[None, None, :] < m, new, old)      # codes seen by step m
        r = Wg.copy()
        for mm in range(M):
            if mm != m:
                r -= C[mm][ctx[:, :, mm]]
        d = C[m][None, None, :, :] - r[:, :, None, :]                 # [N][Gr][256][8]
        if H is None:
            score = np.einsum("nice,nice->nic", d, d)
        else:
            score = np.einsum("nice,ief,nicf->nic", d, H.astype(np.float64), d)
        best = score.min(axis=2)
        chosen = np.take_along_axis(score, new[:, :, m].astype(np.int64)[:, :, None], 2)[:, :, 0]
        assert np.all(chosen <= best + 1e-5 * (1.0 + best)), (m, float(np.max(chosen - best)))


def test_code_update_reduces_error_over_sweeps():
    rng = np.random.default_rng(9)
    N, Gr, M = 128, 16, 2
    books = rng.normal(0, 0.05, size=(M, 256, 8)).astype(np.float16)
    W = rng.normal(0, 0.07, size=(N, Gr * 8)).astype(np.float32)
    codes = np.zeros((N, Gr, M), dtype=np.uint8)
    err = lambda c: float(np.sum((W.astype(np.float64) - O.decode_f64(c, books)) ** 2))
    e0 = err(codes)
    for _ in range(3):
        new = _step(W, books, codes, None, 0, M)
        assert err(new) <= err(codes) + 1e-9
        codes = new
    assert err(codes) < 0.8 * e0
