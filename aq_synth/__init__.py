"""Seeded synthetic inputs for AQ x A8 layers.

This module only draws random arrays with the shapes and value distributions of
the layers the method quantizes (additive-quantized weights, Sec. 2.4 Eq. 4;
8-bit activations, Sec. 4.2.3).  It holds none of the method's arithmetic: no
decode, no quantizer, no contraction.  Both the CPU oracle (tests) and the CUDA
path (tests, bench) consume the arrays it returns, so the two sides always see
identical bytes.

Draw order per layer (one ``numpy.random.default_rng(seed)`` stream, PCG64):
codebooks -> codes -> scale -> bias -> activations.

Array conventions (all C-contiguous numpy arrays):
  codebooks  float16 [M][2**B][g]
  codes      uint8 (B=8) or uint16 (B=16), canonical layout [N][K//g][M]
  scale      float16 [N]            per-output-channel scale
  bias       float16 [N]
  xq         int8 [T][K] (linear) or [Nb][H][W][Cin] (conv, NHWC)
  s_x        python float (per-tensor activation scale, one per timestep)
For a 3x3 convolution the reduction index is k = (kh*3 + kw)*Cin + c (OHWI
weight order) and groups of g consecutive k lie inside one tap.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "LinearSpec", "ConvSpec", "make_linear", "make_conv", "make_f16_activations",
    "WORKLOADS", "SEEDS", "unet_sweep_layers",
]


@dataclass(frozen=True)
class LinearSpec:
    T: int
    K: int
    N: int
    g: int = 8
    M: int = 2
    B: int = 8
    cb_std: float = 0.05
    act: str = "uniform"          # "uniform": U[-127,127]; "normal40": clamp(round(N(0,40)))
    s_x: float = 0.02


@dataclass(frozen=True)
class ConvSpec:
    Nb: int
    H: int
    W: int
    Cin: int
    Cout: int
    stride: int = 1
    pad: int = 1
    kh: int = 3
    kw: int = 3
    g: int = 8
    M: int = 4
    B: int = 8
    cb_std: float = 0.03
    act: str = "normal40"
    s_x: float = 0.02

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.kh) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.kw) // self.stride + 1

    @property
    def K(self) -> int:
        return self.kh * self.kw * self.Cin

    @property
    def T(self) -> int:
        return self.Nb * self.Ho * self.Wo


def _code_dtype(B: int):
    if B == 8:
        return np.uint8
    if B == 16:
        return np.uint16
    raise ValueError(f"B must be 8 or 16, got {B}")


def _weights(rng: np.random.Generator, N: int, K: int, g: int, M: int, B: int,
             cb_std: float):
    codebooks = rng.normal(0.0, cb_std, size=(M, 1 << B, g)).astype(np.float16)
    codes = rng.integers(0, 1 << B, size=(N, K // g, M), dtype=_code_dtype(B))
    scale = rng.uniform(0.5, 1.5, size=N).astype(np.float16)
    bias = rng.normal(0.0, 0.01, size=N).astype(np.float16)
    return codebooks, codes, scale, bias


def _int8_acts(rng: np.random.Generator, shape, kind: str) -> np.ndarray:
    if kind == "uniform":
        return rng.integers(-127, 128, size=shape, dtype=np.int8)
    if kind == "normal40":
        v = np.rint(rng.normal(0.0, 40.0, size=shape))
        return np.clip(v, -127, 127).astype(np.int8)
    raise ValueError(kind)


def make_linear(spec: LinearSpec, seed: int) -> dict:
    """Random AQ linear layer + int8 activations [T][K]."""
    if spec.K % spec.g:
        raise ValueError("K must be a multiple of g")
    rng = np.random.default_rng(seed)
    codebooks, codes, scale, bias = _weights(rng, spec.N, spec.K, spec.g, spec.M,
                                             spec.B, spec.cb_std)
    xq = _int8_acts(rng, (spec.T, spec.K), spec.act)
    return dict(codebooks=codebooks, codes=codes, scale=scale, bias=bias, xq=xq,
                s_x=float(spec.s_x), spec=spec)


def make_conv(spec: ConvSpec, seed: int) -> dict:
    """Random AQ conv layer + NHWC int8 input.  g = 8: groups along Cin inside
    each tap (OHWI); g = 9: one group per (output channel, input channel) 3x3
    filter, codes [Cout][Cin][M] and codebooks [M][2^B][9]."""
    K = spec.K
    if spec.g != 9 and spec.Cin % spec.g:
        raise ValueError("Cin must be a multiple of g")
    rng = np.random.default_rng(seed)
    codebooks, codes, scale, bias = _weights(rng, spec.Cout, K, spec.g, spec.M,
                                             spec.B, spec.cb_std)
    xq = _int8_acts(rng, (spec.Nb, spec.H, spec.W, spec.Cin), spec.act)
    return dict(codebooks=codebooks, codes=codes, scale=scale, bias=bias, xq=xq,
                s_x=float(spec.s_x), spec=spec)


def make_f16_activations(shape, seed: int, std: float = 1.0) -> np.ndarray:
    """Real-valued fp16 activations (input of the 8-bit activation quantizer)."""
    rng = np.random.default_rng(seed)
    return rng.normal(0.0, std, size=shape).astype(np.float16)


# Workloads by name, each drawn from its own seed (SEEDS).
WORKLOADS = {
    # tiny AQ linear, 2x8 codebooks (about 2 bits per weight)
    "tiny_linear": LinearSpec(T=64, K=256, N=256, g=8, M=2, B=8, cb_std=0.05, act="uniform", s_x=0.02),
    # fused qkv projection at the 8x8 level, 32 images x CFG pair: 64*64 tokens
    "qkv": LinearSpec(T=4096, K=960, N=2880, g=8, M=2, B=8, cb_std=0.05, act="uniform", s_x=0.02),
    # 3x3 conv, 16 x 64x64 x 192 -> 192, 4x8 codebooks
    "conv64": ConvSpec(Nb=16, H=64, W=64, Cin=192, Cout=192, stride=1, pad=1, g=8, M=4, B=8,
                cb_std=0.03, act="normal40", s_x=0.02),
    # 3x3 conv, 2 x 8x8 x 960 -> 960, one 2^16-entry codebook
    "conv8_book16": ConvSpec(Nb=2, H=8, W=8, Cin=960, Cout=960, stride=1, pad=1, g=8, M=1,
                             B=16, cb_std=0.05, act="uniform", s_x=0.02),
}
SEEDS = {"tiny_linear": 0, "qkv": 1, "conv64": 2, "conv8_book16": 3}


def unet_sweep_layers():
    """Every AQ conv/linear shape of an LDM-4-ImageNet-like UNet.

    Latent 3x64x64, 192 base channels, channel multipliers (1, 2, 3, 5) giving
    192/384/576/960 channels at resolutions 64/32/16/8, two residual blocks per
    level, 3x3 convs with 1x1 skips where channels change, attention qkv/proj
    linears at 32/16/8.  conv_in / conv_out stay unquantized (Sec. 4.2.1) and
    the time-embedding MLP becomes a table (Sec. 4.2.1), so neither is listed.

    Returns a list of (kind, res, cin, cout, stride, count); kind is "conv3",
    "conv1" or "linear", res the OUTPUT resolution, tokens per image = res**2.
    """
    L = []
    add = L.append
    # level 64 (192 ch)
    add(("conv3", 64, 192, 192, 1, 7))
    add(("conv3", 64, 384, 384, 1, 1))   # up-conv after nearest 2x
    add(("conv3", 64, 384, 192, 1, 2))
    add(("conv3", 64, 576, 192, 1, 1))
    add(("conv1", 64, 384, 192, 1, 2))
    add(("conv1", 64, 576, 192, 1, 1))
    # level 32 (384 ch)
    add(("conv3", 32, 192, 192, 2, 1))   # downsample
    add(("conv3", 32, 192, 384, 1, 1))
    add(("conv3", 32, 384, 384, 1, 6))
    add(("conv3", 32, 576, 576, 1, 1))   # up-conv
    add(("conv3", 32, 576, 384, 1, 1))
    add(("conv3", 32, 768, 384, 1, 1))
    add(("conv3", 32, 960, 384, 1, 1))
    add(("conv1", 32, 192, 384, 1, 1))
    add(("conv1", 32, 576, 384, 1, 1))
    add(("conv1", 32, 768, 384, 1, 1))
    add(("conv1", 32, 960, 384, 1, 1))
    add(("linear", 32, 384, 1152, 1, 5))
    add(("linear", 32, 384, 384, 1, 5))
    # level 16 (576 ch)
    add(("conv3", 16, 384, 384, 2, 1))
    add(("conv3", 16, 384, 576, 1, 1))
    add(("conv3", 16, 576, 576, 1, 6))
    add(("conv3", 16, 960, 960, 1, 1))   # up-conv
    add(("conv3", 16, 960, 576, 1, 1))
    add(("conv3", 16, 1152, 576, 1, 1))
    add(("conv3", 16, 1536, 576, 1, 1))
    add(("conv1", 16, 384, 576, 1, 1))
    add(("conv1", 16, 960, 576, 1, 1))
    add(("conv1", 16, 1152, 576, 1, 1))
    add(("conv1", 16, 1536, 576, 1, 1))
    add(("linear", 16, 576, 1728, 1, 5))
    add(("linear", 16, 576, 576, 1, 5))
    # level 8 (960 ch)
    add(("conv3", 8, 576, 576, 2, 1))
    add(("conv3", 8, 576, 960, 1, 1))
    add(("conv3", 8, 960, 960, 1, 10))
    add(("conv3", 8, 1536, 960, 1, 1))
    add(("conv3", 8, 1920, 960, 1, 2))
    add(("conv1", 8, 576, 960, 1, 1))
    add(("conv1", 8, 1536, 960, 1, 1))
    add(("conv1", 8, 1920, 960, 1, 2))
    add(("linear", 8, 960, 2880, 1, 6))
    add(("linear", 8, 960, 960, 1, 6))
    return L
