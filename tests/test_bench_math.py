"""The roofline arithmetic of bench.py against hand-computed values for the qkv projection
(T=4096, K=960, N=2880, two 8-bit codebooks, g = 8): algorithmic bytes are the packed codes,
the codebooks, the int8 activations read once, the fp16 output and scale + bias."""

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_qkv_algorithmic_bytes_and_flops():
    T, K, N, M, B = 4096, 960, 2880, 2, 8
    codes = N * (K // 8) * M * 1            # one byte per code
    books = M * 256 * 8 * 2                 # fp16 codewords of 8 weights
    acts = T * K                            # int8
    out = T * N * 2                         # fp16
    scale_bias = 2 * N * 2
    assert (codes, books, acts, out, scale_bias) == (691200, 8192, 3932160, 23592960, 11520)
    assert bench.alg_bytes(T, K, N, M, B) == codes + books + acts + out + scale_bias == 28236032
    assert bench.linear_flops(T, N, K) == 2 * 4096 * 2880 * 960 == 22649241600


def test_alg_bytes_formats():
    # one 2^16-entry codebook: 16-bit codes, 65536 codewords; fp32 output
    T, K, N = 128, 8640, 960
    assert bench.alg_bytes(T, K, N, 1, 16, out_bytes=4) == (
        N * (K // 8) * 2 + 65536 * 8 * 2 + T * K + T * N * 4 + 4 * N)
