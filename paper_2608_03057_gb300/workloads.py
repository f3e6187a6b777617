"""Seeded synthetic inputs and layer inventories for the masked-W8A8 path.

This module holds no arithmetic of the method: it only draws random numbers
(numpy PCG64, fixed seeds) and lists layer shapes.  Both the CUDA path and the
CPU oracle are fed from here, so the two always see identical bytes.

Shapes follow the three backbones the paper evaluates (Sec. 4.1; App. D.3
gives the quantized-tensor counts 224 / 160 / 560), with random weights in
place of the trained checkpoints, which are not available:
  * PixArt-Sigma at 1024 px: 4096 image tokens, 300 text tokens, hidden 1152,
    28 blocks x 8 quantized linears = 224 tensors.
  * SANA-1.6B at 1024 px: batch 4 x 1024 tokens, 4 x 300 text tokens, hidden
    2240, 20 blocks x 8 quantized linears = 160 tensors.
  * SDXL-Turbo at 512 px: 64x64 latent, 77 text tokens; 70 transformer blocks
    (10 at width 640 on 32x32, 60 at width 1280 on 16x16) x 8 linears = 560
    tensors, plus 34 3x3 convs (10 at 320@64x64, 10 at 640@32x32,
    14 at 1280@16x16).
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np

LINEAR = 0
CONV3X3 = 1


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


@dataclasses.dataclass(frozen=True)
class Layer:
    name: str
    kind: int          # LINEAR or CONV3X3
    M: int             # tokens (linear) or B*H*W output pixels (conv)
    N: int             # output features / Cout
    K: int             # input features / 9*Cin
    H: int = 0         # conv only
    W: int = 0
    Cin: int = 0
    B: int = 1

    @property
    def ops(self) -> int:
        """Multiply-add count x 2 (int8-equivalent ops of one call)."""
        return 2 * self.M * self.N * self.K


def normal(shape, seed: int, std: float = 1.0, dtype=np.float32) -> np.ndarray:
    return (rng(seed).standard_normal(shape) * std).astype(dtype)


def uniform_codes(shape, seed: int, lo: int = -127, hi: int = 127) -> np.ndarray:
    return rng(seed).integers(lo, hi + 1, size=shape, dtype=np.int64).astype(np.int8)


def uniform(shape, seed: int, lo: float, hi: float) -> np.ndarray:
    return rng(seed).uniform(lo, hi, size=shape).astype(np.float32)


def device_normal(shape, seed: int, std: float = 1.0, dtype=None, device="cuda"):
    """N(0, std^2) drawn on the GPU with torch's seeded Philox generator (for
    benchmark-sized tensors that would take too long to draw on the host)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t if dtype is None else t.to(dtype)


# ----------------------------------------------------------------------------
# Layer inventories
# ----------------------------------------------------------------------------

def single_linear() -> List[Layer]:
    """One 1152x1152 linear on 256 tokens."""
    return [Layer("linear", LINEAR, 256, 1152, 1152)]


def pixart_sigma(blocks: int = 28, tokens: int = 4096, text: int = 300, hidden: int = 1152) -> List[Layer]:
    out = []
    for i in range(blocks):
        h = hidden
        out += [
            Layer(f"b{i}.attn.qkv", LINEAR, tokens, 3 * h, h),
            Layer(f"b{i}.attn.proj", LINEAR, tokens, h, h),
            Layer(f"b{i}.cross.q", LINEAR, tokens, h, h),
            Layer(f"b{i}.cross.k", LINEAR, text, h, h),
            Layer(f"b{i}.cross.v", LINEAR, text, h, h),
            Layer(f"b{i}.cross.out", LINEAR, tokens, h, h),
            Layer(f"b{i}.mlp.fc1", LINEAR, tokens, 4 * h, h),
            Layer(f"b{i}.mlp.fc2", LINEAR, tokens, h, 4 * h),
        ]
    return out


def sana_1600m(blocks: int = 20, tokens: int = 4 * 1024, text: int = 4 * 300, hidden: int = 2240,
               mlp: int = 5600) -> List[Layer]:
    out = []
    for i in range(blocks):
        h = hidden
        out += [
            Layer(f"b{i}.attn.qkv", LINEAR, tokens, 3 * h, h),
            Layer(f"b{i}.attn.proj", LINEAR, tokens, h, h),
            Layer(f"b{i}.cross.q", LINEAR, tokens, h, h),
            Layer(f"b{i}.cross.k", LINEAR, text, h, h),
            Layer(f"b{i}.cross.v", LINEAR, text, h, h),
            Layer(f"b{i}.cross.out", LINEAR, tokens, h, h),
            Layer(f"b{i}.glu.up", LINEAR, tokens, 2 * mlp, h),
            Layer(f"b{i}.glu.down", LINEAR, tokens, h, mlp),
        ]
    return out


def _sdxl_block(prefix: str, C: int, M: int, text: int = 77, ctx: int = 2048) -> List[Layer]:
    return [
        Layer(f"{prefix}.attn1.qkv", LINEAR, M, 3 * C, C),
        Layer(f"{prefix}.attn1.out", LINEAR, M, C, C),
        Layer(f"{prefix}.attn2.q", LINEAR, M, C, C),
        Layer(f"{prefix}.attn2.k", LINEAR, text, C, ctx),
        Layer(f"{prefix}.attn2.v", LINEAR, text, C, ctx),
        Layer(f"{prefix}.attn2.out", LINEAR, M, C, C),
        Layer(f"{prefix}.ff.geglu", LINEAR, M, 8 * C, C),
        Layer(f"{prefix}.ff.out", LINEAR, M, C, 4 * C),
    ]


def _conv(name: str, C: int, H: int, W: int, B: int = 1) -> Layer:
    return Layer(name, CONV3X3, B * H * W, C, 9 * C, H=H, W=W, Cin=C, B=B)


def sdxl_turbo() -> List[Layer]:
    """Depth-ordered: down path, middle, up path."""
    out: List[Layer] = []
    # down 320 @ 64x64: conv_in + 2 resnets (2 convs each) + downsample
    out += [_conv(f"down0.conv{i}", 320, 64, 64) for i in range(5)]
    # down 640 @ 32x32: 2 resnets with 2 transformer blocks each
    out += [_conv(f"down1.conv{i}", 640, 32, 32) for i in range(5)]
    for r in range(2):
        for t in range(2):
            out += _sdxl_block(f"down1.r{r}.t{t}", 640, 1024)
    # down 1280 @ 16x16: 2 resnets, 10 transformer blocks each
    out += [_conv(f"down2.conv{i}", 1280, 16, 16) for i in range(4)]
    for r in range(2):
        for t in range(10):
            out += _sdxl_block(f"down2.r{r}.t{t}", 1280, 256)
    # middle: 2 resnets around 10 transformer blocks
    out += [_conv(f"mid.conv{i}", 1280, 16, 16) for i in range(4)]
    for t in range(10):
        out += _sdxl_block(f"mid.t{t}", 1280, 256)
    # up 1280 @ 16x16: 3 resnets with 10 blocks each
    out += [_conv(f"up0.conv{i}", 1280, 16, 16) for i in range(6)]
    for r in range(3):
        for t in range(10):
            out += _sdxl_block(f"up0.r{r}.t{t}", 1280, 256)
    # up 640 @ 32x32: 3 resnets with 2 blocks each
    for r in range(3):
        for t in range(2):
            out += _sdxl_block(f"up1.r{r}.t{t}", 640, 1024)
    out += [_conv(f"up1.conv{i}", 640, 32, 32) for i in range(5)]
    out += [_conv(f"up2.conv{i}", 320, 64, 64) for i in range(5)]
    return out


# Layers that read the same input tensor: the key and value projections of a
# cross-attention both take the text tokens.
SHARED_INPUT_PAIRS = ((".cross.k", ".cross.v"), (".attn2.k", ".attn2.v"))


def input_groups(layers: List[Layer]) -> List[List[int]]:
    """The inventory as units of layers that read one input: a cross-attention's
    key and value projections form a unit of two (consecutive, same M and K),
    every other layer a unit of its own.  Indices follow the inventory."""
    out: List[List[int]] = []
    i = 0
    while i < len(layers):
        l = layers[i]
        if i + 1 < len(layers):
            m = layers[i + 1]
            for a, b in SHARED_INPUT_PAIRS:
                if (l.name.endswith(a) and m.name.endswith(b) and l.name[:-len(a)] == m.name[:-len(b)]
                        and (l.M, l.K, l.kind) == (m.M, m.K, m.kind)):
                    out.append([i, i + 1])
                    i += 2
                    break
            else:
                out.append([i])
                i += 1
            continue
        out.append([i])
        i += 1
    return out


# Layers that read the text tokens: the key and value projections of every
# cross-attention block.  In all three networks the text embedding is computed once
# per forward pass and is the same tensor for every block.
TEXT_INPUT_SUFFIXES = (".cross.k", ".cross.v", ".attn2.k", ".attn2.v")
MAX_SHARED_MEMBERS = 256


def shared_input_units(layers: List[Layer], max_members: int = MAX_SHARED_MEMBERS) -> List[List[int]]:
    """The inventory as units of layers that read one input, with every layer that
    reads the text tokens gathered into units of one shape (kind, M, N, K) each, at
    most max_members layers per unit, in inventory order within a unit.  These units
    come first (their input does not depend on the image tokens, so they can run
    before any block); every other layer is a unit of its own, in inventory order."""
    shared = {}
    rest: List[List[int]] = []
    for i, l in enumerate(layers):
        if l.name.endswith(TEXT_INPUT_SUFFIXES):
            shared.setdefault((l.kind, l.M, l.N, l.K), []).append(i)
        else:
            rest.append([i])
    units: List[List[int]] = []
    for members in shared.values():  # shapes in order of first appearance
        for j in range(0, len(members), max_members):
            units.append(members[j:j + max_members])
    return units + rest


def sweep_shapes():
    """GEMM sweep: M x (K = N) x b."""
    for M in (1024, 4096, 16384):
        for KN in (1152, 2240, 4096):
            yield M, KN


# ----------------------------------------------------------------------------
# Bit schedules (uint8 [L][S], values 2..8)
# ----------------------------------------------------------------------------

def schedule_uniform(L: int, S: int, bits, seed: int, edge_stages: int = 0, edge_p8: float = 0.5) -> np.ndarray:
    """Per-(layer, stage) bits drawn uniformly from `bits`; in the first and last
    `edge_stages` stages a draw is replaced by 8 with probability `edge_p8`."""
    g = rng(seed)
    bits = np.asarray(sorted(bits), np.uint8)
    tab = bits[g.integers(0, len(bits), size=(L, S))]
    if edge_stages:
        edge = list(range(edge_stages)) + list(range(S - edge_stages, S))
        coin = g.random((L, len(edge))) < edge_p8
        for j, s in enumerate(edge):
            tab[coin[:, j], s] = 8
    return np.ascontiguousarray(tab, dtype=np.uint8)


def schedule_constant(L: int, S: int, b: int) -> np.ndarray:
    return np.full((L, S), b, np.uint8)


def schedule_for(config: str, L: int, seed: int = 7) -> np.ndarray:
    if config in ("pixart", "pixart_lr"):
        return schedule_uniform(L, 20, (3, 4, 5, 6, 8), seed, edge_stages=2)
    if config == "sana":
        return schedule_uniform(L, 20, (2, 3, 4, 6, 8), seed)
    if config == "sdxl":
        return schedule_uniform(L, 4, (4, 5, 6, 8), seed)
    if config == "pixart_a4":
        # 4-bit activations at the W4A4 computational budget: operating precisions
        # averaging 4 bits (the quality table's W4A4-budget row has Eff. W 3.98)
        return schedule_uniform(L, 20, (2, 3, 4, 5, 6), seed)
    if config == "single":
        return np.array([[8, 6, 4, 3]], np.uint8)
    if config == "sweep":
        return np.array([[2, 3, 4, 5, 6, 7, 8, 8]], np.uint8)
    raise KeyError(config)


def inventory_blocks(config: str, blocks: int) -> List[Layer]:
    """The first `blocks` transformer blocks of a DiT inventory (small cases)."""
    if config in ("pixart", "pixart_a4", "pixart_lr"):
        return pixart_sigma(blocks=blocks)
    if config == "sana":
        return sana_1600m(blocks=blocks)
    return inventory(config)


def inventory(config: str) -> List[Layer]:
    return {"single": single_linear, "pixart": pixart_sigma, "pixart_a4": pixart_sigma, "pixart_lr": pixart_sigma,
            "sana": sana_1600m, "sdxl": sdxl_turbo}[config]()


# Activation precision n of each workload (8 unless listed).
ACT_BITS = {"pixart_a4": 4}
# Rank of the 16-bit low-rank branch beside every linear layer (SVDQuant+TASQ: a
# frozen SVD branch of rank 32 in the 4-bit setting, 16 in the 6-bit one), or 0.
LOWRANK = {"pixart_lr": 32}


# ----------------------------------------------------------------------------
# Per-layer tensors
# ----------------------------------------------------------------------------

def layer_weight(layer: Layer, seed: int, std: float = 0.02) -> np.ndarray:
    """Float weights [N][K] (conv: [Cout][3][3][Cin] flattened to K = 9*Cin)."""
    return normal((layer.N, layer.K), seed, std)


def layer_bias(layer: Layer, seed: int, std: float = 0.02) -> np.ndarray:
    return normal((layer.N,), seed, std)


def layer_input(layer: Layer, seed: int, dtype=np.float32) -> np.ndarray:
    """Float activations: [M][K] for a linear, NHWC [B][H][W][Cin] for a conv."""
    if layer.kind == CONV3X3:
        return normal((layer.B, layer.H, layer.W, layer.Cin), seed, 1.0, dtype)
    return normal((layer.M, layer.K), seed, 1.0, dtype)
