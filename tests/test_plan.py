"""CPU checks of the tensor-core route's launch planning (tasq_plan_tc): the
tile configuration, token tiling, K split and grid that a contraction of a
given shape gets.  The plan is host logic and needs no GPU; the GPU suite
checks that the launches follow it (kernel counts).

The rules checked here:
  - tiles are 128 output channels by 64, 192 or 256 tokens; 256-token tiles
    keep one accumulator in tensor memory, the others two;
  - 256-token tiles exactly when the 192-token tiling needs more than one wave
    of CTAs and the 256-token tiling fits in one; 64-token tiles when the
    192-token tiles would leave at least half of the SMs idle;
  - a convolution tiles each image into boxes of whole rows of 2^j pixels
    (2^j >= min(W, 64)), one box per tile;
  - K is split only for two-accumulator tiles that leave half of the SMs idle,
    into as many slices as fit the SMs, at most 16, each at least 8 blocks of
    128 K, and only as far as the context's 32 MB split scratch holds
    splits * M * N int32 partial sums;
  - the contraction is persistent: min(tiles * splits, SMs) CTAs.
"""
import ctypes
import math
import os
import shutil
import subprocess

import pytest

from paper_2608_03057_gb300 import tasq, workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SMS = 152  # GB300
SPLIT_CAP = (32 << 20) // 4


@pytest.fixture(scope="module", autouse=True)
def built_lib():
    from paper_2608_03057_gb300 import build
    return build.build()


def plan(kind, M=0, N=0, K=0, B=0, H=0, W=0, Cin=0, sms=SMS):
    return tasq.tasq_plan_tc(kind, M, N, K, B, H, W, Cin, sms)


def linear(M, N, K, sms=SMS):
    return plan(tasq.TASQ_LINEAR, M, N, K, sms=sms)


def conv(B, H, W, Cin, Cout, sms=SMS):
    return plan(tasq.TASQ_CONV3X3, 0, Cout, 0, B, H, W, Cin, sms=sms)


def token_tiles(bt, M, B=0, H=0, W=0):
    """Token tiles of a bt-token tiling (linear: runs of bt tokens; conv: boxes
    of bt / 2^j rows x 2^j pixels per image)."""
    if not W:
        return math.ceil(M / bt), 0, 0
    cols = 1
    while cols < W and cols < 64:
        cols *= 2
    rows = bt // cols
    return B * math.ceil(H / rows) * math.ceil(W / cols), rows, cols


def check_rules(p, M, N, K, sms=SMS, B=0, H=0, W=0):
    assert p["tile_channels"] == 128
    assert p["tiles_ch"] == math.ceil(N / 128)
    if M == 0:
        assert p["kernels"] == 0 and p["grid"] == 0
        return
    std = p["tiles_ch"] * token_tiles(192, M, B, H, W)[0]
    wide = p["tiles_ch"] * token_tiles(256, M, B, H, W)[0]
    if std > sms and wide <= sms:
        assert (p["tile_tokens"], p["acc_buffers"]) == (256, 1)
    elif 2 * std <= sms:
        assert (p["tile_tokens"], p["acc_buffers"]) == (64, 2)
    else:
        assert (p["tile_tokens"], p["acc_buffers"]) == (192, 2)
    tok, rows, cols = token_tiles(p["tile_tokens"], M, B, H, W)
    assert p["tiles_tok"] == tok
    assert (p["box_rows"], p["box_cols"]) == (rows, cols)
    if W:
        assert rows * cols == p["tile_tokens"] and (cols >= W or cols == 64)
    tiles = p["tiles_ch"] * tok
    # every output is in exactly one tile: the tiles cover M tokens, ragged edges included
    if not W:
        assert (tok - 1) * p["tile_tokens"] < M <= tok * p["tile_tokens"]
    S = 1
    if p["acc_buffers"] == 2 and 2 * tiles <= sms:
        S = min(sms // tiles, math.ceil(K / 128) // 8, 16, SPLIT_CAP // (M * N))
        S = S if S >= 2 else 1
    assert p["splits"] == S
    assert p["grid"] == min(tiles * S, sms)
    assert p["kernels"] == (2 if S > 1 else 1)
    if S > 1:
        assert p["tile_tokens"] == 64
        assert S * 8 * 128 <= math.ceil(K / 128) * 128 and S * M * N <= SPLIT_CAP
        assert p["reduce_grid"] == min(math.ceil(M * (N // 4) / 256), 8 * sms)
    else:
        assert p["reduce_grid"] == 0


def test_struct_layout_matches_header(tmp_path):
    """The binding's ctypes struct has the C struct's size and field offsets."""
    cc = shutil.which("gcc") or shutil.which("cc")
    if not cc:
        pytest.skip("no C compiler")
    fields = [name for name, _ in tasq.tasq_tc_plan._fields_]
    src = tmp_path / "layout.c"
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "tasq.h"\nint main(void) {\n'
                   '  printf("%zu\\n", sizeof(tasq_tc_plan));\n'
                   + "".join(f'  printf("%zu\\n", offsetof(tasq_tc_plan, {f}));\n' for f in fields) + "  return 0;\n}\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    assert got[0] == ctypes.sizeof(tasq.tasq_tc_plan)
    assert got[1:] == [getattr(tasq.tasq_tc_plan, f).offset for f in fields]


@pytest.mark.parametrize("config", ["pixart", "sana", "sdxl"])
def test_every_layer_of_the_workloads(config):
    """Each layer of the three workloads' inventories, on 152 SMs."""
    for l in workloads.inventory(config):
        if l.kind == workloads.CONV3X3:
            p = conv(l.B, l.H, l.W, l.Cin, l.N)
            check_rules(p, l.B * l.H * l.W, l.N, 9 * l.Cin, B=l.B, H=l.H, W=l.W)
        else:
            check_rules(linear(l.M, l.N, l.K), l.M, l.N, l.K)


def test_worked_plans():
    """Plans worked out by hand for a few layers of the workloads."""
    # PixArt-Sigma qkv at 1024 px: 27 x 22 192-token tiles (27 x 16 = 432 256-token
    # tiles are still more than one wave): persistent over all 152 SMs
    p = linear(4096, 3456, 1152)
    assert (p["tile_tokens"], p["tiles_ch"], p["tiles_tok"], p["splits"], p["grid"], p["kernels"]) == \
        (192, 27, 22, 1, 152, 1)
    # cross-attention keys and values over 300 text tokens: 18 x 2 = 36 192-token tiles
    # would leave 116 SMs idle, so 18 x 5 64-token tiles; 9 K blocks cannot be split
    p = linear(300, 2304, 1152)
    assert (p["tile_tokens"], p["tiles_tok"], p["splits"], p["grid"]) == (64, 5, 1, 90)
    # a 4000 x 1096 output: 9 x 21 = 189 192-token tiles, 9 x 16 = 144 256-token tiles
    p = linear(4000, 1096, 384)
    assert (p["tile_tokens"], p["acc_buffers"], p["tiles_tok"], p["grid"]) == (256, 1, 16, 144)
    # few tokens, long K: 9 tiles, 36 K blocks -> 4 slices of 9 blocks; the
    # reduction covers 64 x 1152 / 4 = 18432 four-channel groups in 72 blocks
    p = linear(64, 1152, 4608)
    assert (p["tile_tokens"], p["tiles_ch"], p["splits"], p["grid"], p["reduce_grid"], p["kernels"]) == \
        (64, 9, 4, 36, 72, 2)
    # SDXL 3x3 conv at 64 x 64, 640 channels: boxes of 3 rows x 64 pixels
    p = conv(1, 64, 64, 640, 640)
    assert (p["tile_tokens"], p["box_rows"], p["box_cols"], p["tiles_tok"], p["tiles_ch"]) == (192, 3, 64, 22, 5)
    assert p["grid"] == 110 and p["splits"] == 1  # 110 tiles: under one wave, but 2 x 110 > 152
    # a 6 x 6 image, 64 channels: 8-pixel rows, 8 rows per 64-token box; K = 576 is
    # 5 K blocks, too few to split
    p = conv(2, 6, 6, 64, 128)
    assert (p["tile_tokens"], p["box_rows"], p["box_cols"], p["tiles_tok"], p["splits"], p["grid"]) == \
        (64, 8, 8, 2, 1, 2)


@pytest.mark.parametrize("sms", [1, 2, 8, 76, 132, 148, 152, 160])
def test_rules_hold_for_any_sm_count(sms):
    shapes = [(4096, 3456, 1152), (4096, 1152, 4608), (300, 1152, 1168), (77, 640, 2048), (64, 128, 4096),
              (4000, 1096, 384), (1, 8, 16), (16384, 4096, 4096), (8192, 2240, 2240), (1200, 4480, 2240)]
    for M, N, K in shapes:
        check_rules(linear(M, N, K, sms), M, N, K, sms)
    for B, H, W, Cin, Cout in [(1, 128, 128, 320, 320), (2, 32, 32, 1280, 1280), (3, 5, 7, 64, 136),
                               (1, 1, 1, 64, 8), (1, 200, 100, 128, 64)]:
        check_rules(conv(B, H, W, Cin, Cout, sms), B * H * W, Cout, 9 * Cin, sms, B, H, W)


def test_split_limits():
    """Which limit sets the slice count.  Splitting only happens with 64-token
    tiles, whose partial sums take at most 8192 int32 per tile and slice, so on
    152 SMs the 32 MB scratch never binds before the SM count or the 16-slice
    limit; on a device with ten times as many SMs it does."""
    # 4 tiles, 64 K blocks: 8 slices of 8 blocks (38 would fit the SMs)
    p = linear(64, 512, 8192)
    assert (p["splits"], p["grid"]) == (8, 32)
    # 1 tile, 256 K blocks: the 16-slice limit
    p = linear(64, 128, 32768)
    assert (p["splits"], p["grid"]) == (16, 16)
    # 64 tiles: 152 // 64 = 2 slices
    p = linear(64, 8192, 8192)
    assert (p["splits"], p["grid"]) == (2, 128)
    check_rules(p, 64, 8192, 8192)
    # 100 tiles of 64 x 128 on 1600 SMs: 16 slices would fit the SMs and K, but
    # 16 x 640 x 1280 partial sums exceed 2^23, so 10 slices
    p = linear(640, 1280, 16384, sms=1600)
    assert (p["tile_tokens"], p["splits"], p["grid"]) == (64, 10, 1000)
    assert 10 * 640 * 1280 <= SPLIT_CAP < 11 * 640 * 1280
    check_rules(p, 640, 1280, 16384, sms=1600)
    # 192-token tiles are chosen only when twice their count exceeds the SMs, and
    # 256-token tiles only beyond one wave, so neither is ever split
    # 64 192-token tiles would leave half the SMs idle: 192 64-token tiles instead,
    # more than one wave, so K is not split
    p = linear(192 * 8, 1024, 16384)
    assert (p["tile_tokens"], p["tiles_tok"], p["splits"], p["grid"]) == (64, 24, 1, 152)
    p = linear(192 * 10, 1024, 16384)  # 80 192-token tiles
    assert (p["tile_tokens"], p["splits"], p["grid"]) == (192, 1, 80)


def test_empty_token_dimension():
    p = linear(0, 1152, 1152)
    assert p["kernels"] == 0 and p["grid"] == 0 and p["tiles_ch"] == 9
    p = conv(0, 16, 16, 64, 64)
    assert p["kernels"] == 0 and p["grid"] == 0


@pytest.mark.parametrize("args,code", [
    ((tasq.TASQ_LINEAR, 64, 128, 1000), tasq.TASQ_ERR_UNSUPPORTED),   # K % 16
    ((tasq.TASQ_LINEAR, 64, 100, 1024), tasq.TASQ_ERR_UNSUPPORTED),   # N % 8
    ((tasq.TASQ_LINEAR, -1, 128, 1024), tasq.TASQ_ERR_INVALID_ARG),
    ((tasq.TASQ_LINEAR, 64, 0, 1024), tasq.TASQ_ERR_INVALID_ARG),
    ((7, 64, 128, 1024), tasq.TASQ_ERR_INVALID_ARG),                  # kind
    ((tasq.TASQ_CONV3X3, 0, 64, 0, 1, 8, 8, 32), tasq.TASQ_ERR_UNSUPPORTED),   # Cin % 64 on this route
    ((tasq.TASQ_CONV3X3, 0, 64, 0, 1, 8, 8, 40), tasq.TASQ_ERR_UNSUPPORTED),   # Cin % 16
    ((tasq.TASQ_CONV3X3, 0, 64, 0, 1, 0, 8, 64), tasq.TASQ_ERR_INVALID_ARG),   # H
])
def test_rejected_shapes(args, code):
    full = list(args) + [0] * (8 - len(args))
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_plan_tc(*full, SMS)
    assert e.value.code == code
    with pytest.raises(tasq.TasqError) as e:
        tasq.tasq_plan_tc(tasq.TASQ_LINEAR, 64, 128, 1024, 0, 0, 0, 0, 0)
    assert e.value.code == tasq.TASQ_ERR_INVALID_ARG


def test_input_groups_pair_cross_attention_keys_and_values():
    """The benchmark's units: each cross-attention's key and value projections
    (same block, same input shape) share one input; nothing else is grouped."""
    from paper_2608_03057_gb300 import workloads
    for name, pairs in (("pixart", 28), ("sana", 20), ("sdxl", 70), ("single", 0)):
        layers = workloads.inventory(name)
        units = workloads.input_groups(layers)
        assert sorted(i for u in units for i in u) == list(range(len(layers)))
        two = [u for u in units if len(u) == 2]
        assert len(two) == pairs
        for a, b in two:
            la, lb = layers[a], layers[b]
            assert b == a + 1 and (la.M, la.K) == (lb.M, lb.K)
            assert la.name.rsplit(".", 1)[1] == "k" and lb.name.rsplit(".", 1)[1] == "v"
            assert la.name.rsplit(".", 1)[0] == lb.name.rsplit(".", 1)[0]


def test_shared_input_units_gather_every_text_projection():
    """The benchmark's default units: every layer that reads the text tokens (the key
    and value projections of all cross-attention blocks) in one unit per shape, at
    most 256 layers, placed first; every other layer alone, in inventory order."""
    from paper_2608_03057_gb300 import workloads
    for name, sizes in (("pixart", [56]), ("sana", [40]), ("sdxl", [20, 120]), ("single", [])):
        layers = workloads.inventory(name)
        units = workloads.shared_input_units(layers)
        assert sorted(i for u in units for i in u) == list(range(len(layers)))
        shared = [u for u in units if len(u) > 1]
        assert [len(u) for u in shared] == sizes
        assert units[:len(shared)] == shared
        for u in shared:
            assert all(layers[i].name.rsplit(".", 1)[1] in ("k", "v") for i in u)
            assert len({(layers[i].kind, layers[i].M, layers[i].N, layers[i].K) for i in u}) == 1
            assert u == sorted(u)
        rest = [u[0] for u in units[len(shared):]]
        assert rest == sorted(rest) and all(len(u) == 1 for u in units[len(shared):])
        assert not any(layers[i].name.endswith(workloads.TEXT_INPUT_SUFFIXES) for i in rest)
    layers = workloads.inventory("sdxl")
    assert [len(u) for u in workloads.shared_input_units(layers, 50) if len(u) > 1] == [20, 50, 50, 20]
