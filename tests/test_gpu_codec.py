"""GPU parity of the integer/byte kernels, bit-exact against the oracle:
activation quantizer, code packing, and the AQ decode rule."""

import numpy as np
import pytest

from aq_synth import SEEDS, WORKLOADS, LinearSpec, make_f16_activations, make_conv, make_linear
from oracle import aq_oracle as O

from gpu_util import dev, pack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2506_05960_gb300 as aq
    aq.load_library()


@pytest.mark.parametrize("numel", [1, 15, 16, 17, 4096 + 7, 1_000_003])
@pytest.mark.parametrize("s_x", [0.02, 0.5, 3.0])
def test_quant_act_bit_exact(numel, s_x):
    import torch
    import paper_2506_05960_gb300 as aq
    x = make_f16_activations((numel,), seed=numel, std=2.0)
    xq = torch.full((numel + 16,), 99, dtype=torch.int8, device="cuda")
    aq.aq_quant_act(dev(x), xq, numel, s_x)
    got = xq.cpu().numpy()
    assert np.array_equal(got[:numel], O.quant_act(x, s_x))
    assert np.all(got[numel:] == 99)          # nothing written past numel


def test_quant_act_special_values():
    import torch
    import paper_2506_05960_gb300 as aq
    vals = [0.0, -0.0, np.inf, -np.inf, np.nan, 65504.0, -65504.0, 1.25, 1.75, -1.25, 0.25,
            -0.25, 63.5, -63.75, 6e-8, -6e-8]
    x = np.array(vals * 3, dtype=np.float16)
    xq = torch.empty(x.size, dtype=torch.int8, device="cuda")
    aq.aq_quant_act(dev(x), xq, x.size, 0.5)
    assert np.array_equal(xq.cpu().numpy(), O.quant_act(x, 0.5))


@pytest.mark.parametrize("s_x", [0.05, 0.02, 0.1, 0.125, 1.0, 0.0473, 0.0387, 7.3e-3,
                                 1.1920929e-07, 300.0])
def test_quant_act_every_f16_value(s_x):
    """All 65536 fp16 bit patterns (ties of x / s are exact for scales with few
    significant bits, e.g. 0.05 at x = 0.875), bit-exact against the rule."""
    import torch
    import paper_2506_05960_gb300 as aq
    x = np.arange(65536, dtype=np.uint16).view(np.float16)
    x = np.concatenate([x, x[::-1]])          # each value in several lanes / positions
    xq = torch.empty(x.size, dtype=torch.int8, device="cuda")
    aq.aq_quant_act(dev(x), xq, x.size, float(np.float32(s_x)))
    assert np.array_equal(xq.cpu().numpy(), O.quant_act(x, float(np.float32(s_x))))


@pytest.mark.parametrize("N,K,M,B", [(256, 256, 2, 8), (37, 200, 3, 8), (8, 64, 8, 8),
                                     (960, 8640, 1, 16), (24, 72, 2, 16), (5, 8, 1, 8)])
def test_pack_bit_exact(N, K, M, B):
    rng = np.random.default_rng(N + K)
    dt = np.uint8 if B == 8 else np.uint16
    codes = rng.integers(0, 1 << B, size=(N, K // 8, M), dtype=dt)
    got = pack(codes, N, K, M, B).cpu().numpy()
    assert np.array_equal(got, O.pack_codes(codes, 8))


def _decode_gpu(codes, books, N, K, M, B):
    import torch
    import paper_2506_05960_gb300 as aq
    packed = pack(codes, N, K, M, B)
    W = torch.full((N, K), float("nan"), dtype=torch.float16, device="cuda")
    aq.aq_decode(packed, dev(books), W, N, K, 8, M, B)
    return W.cpu().numpy()


@pytest.mark.parametrize("wl", ["tiny_linear", "qkv", "conv64", "conv8_book16"])
def test_decode_bit_exact_workloads(wl):
    spec = WORKLOADS[wl]
    make = make_linear if isinstance(spec, LinearSpec) else make_conv
    inp = make(spec, seed=SEEDS[wl])
    N, G, M = inp["codes"].shape
    B = spec.B
    W = _decode_gpu(inp["codes"], inp["codebooks"], N, G * 8, M, B)
    ref = O.decode_rule_f16(inp["codes"], inp["codebooks"])
    assert np.array_equal(W.view(np.uint16), ref.view(np.uint16))


@pytest.mark.parametrize("M", [1, 2, 3, 4, 8])
def test_decode_edge_values(M):
    """Overflow to +-inf, subnormals, signed zeros, codes 0 and 255, ragged K."""
    rng = np.random.default_rng(M)
    books = np.zeros((M, 256, 8), dtype=np.float16)
    special = np.array([65504, -65504, 32768, 6e-8, -6e-8, 0.0, -0.0, 1.0, 2 ** -14, 1e-5],
                       dtype=np.float16)
    books[:] = special[rng.integers(0, special.size, size=books.shape)]
    books[:, 0, :] = np.float16(-0.0)
    books[:, 255, :] = np.float16(65504)
    N, K = 40, 200
    codes = rng.integers(0, 256, size=(N, K // 8, M), dtype=np.uint8)
    codes[0, :, :] = 0
    codes[1, :, :] = 255
    W = _decode_gpu(codes, books, N, K, M, 8)
    ref = O.decode_rule_f16(codes, books)
    assert np.array_equal(W.view(np.uint16), ref.view(np.uint16))
    if M >= 2:
        assert np.isinf(ref[1]).all()           # 65504 + 65504 overflows
    assert (ref[0].view(np.uint16) == 0x8000).all()   # -0 + ... + -0 = -0


def test_decode_16bit_codes_extremes():
    rng = np.random.default_rng(16)
    books = rng.normal(0, 0.05, size=(2, 1 << 16, 8)).astype(np.float16)
    N, K = 16, 136
    codes = rng.integers(0, 1 << 16, size=(N, K // 8, 2), dtype=np.uint16)
    codes[0] = 0
    codes[1] = 65535
    W = _decode_gpu(codes, books, N, K, 2, 16)
    assert np.array_equal(W.view(np.uint16), O.decode_rule_f16(codes, books).view(np.uint16))
