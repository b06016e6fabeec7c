"""Other group shapes (Sec. 2.1 with g_out x g_in groups; the Sec. 3.5 ablation
and App. E evaluate square 16x16 .. 128x128): the CUDA path against the oracle,
through the C ABI.

Packing and unpacking must match the oracle's pack_groups / unpack_groups bit
for bit; y must satisfy |y - y_oracle| <= 2^-7 * sum_kept |x w| + 1e-6 per
element, with the oracle's y and magnitude sum for the same group shape.
"""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl
from tests._gpu_util import REL, ABS, bf16_to_f64, sample_tokens, to_bits, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


def make(gs, out, inp, g, d, seed):
    import torch
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    B = wl.random_mask(out // g, inp // g, d, seed=seed + 500)
    return Wb, B, gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), g, g)


def check_y(y_bits, xb, Wb, B, g, tokens=None, what=""):
    if tokens is None:
        yr, A = orc.linear(xb, Wb, B, g, g)
        yg = bf16_to_f64(y_bits)
    else:
        yr, A = orc.linear_tokens(xb, Wb, B, tokens, g, g)
        yg = bf16_to_f64(y_bits[np.asarray(tokens)])
    err = np.abs(yg - yr)
    bad = err > REL * A + ABS
    assert not bad.any(), f"{what}: {int(bad.sum())} elements outside the bound, first at {tuple(np.argwhere(bad)[0])}"


SHAPES = [(48, 64, 0.5, 1), (128, 128, 0.5, 2), (256, 512, 0.3, 3), (1024, 1024, 0.5, 4), (4096, 4096, 0.5, 5),
          (11008, 4096, 0.45, 6), (4096, 11008, 0.5, 7), (512, 3584, 0.7, 8), (640, 256, 1.0, 9), (384, 768, 0.0, 10)]


@pytest.mark.parametrize("g", [16, 32, 64, 128])
@pytest.mark.parametrize("out,inp,d,seed", SHAPES)
def test_pack_and_unpack_are_bit_exact(gs, g, out, inp, d, seed):
    if out % g or inp % g:
        pytest.skip("shape not tiled by the group")
    Wb, B, p = make(gs, out, inp, g, d, seed)
    ref = orc.pack_groups(Wb, B, g, g)
    got = p.export()
    assert np.array_equal(got["offsets"], ref.offsets)
    assert np.array_equal(got["row_idx"], ref.block_row)
    assert np.array_equal(got["tiles"], ref.tiles)
    assert p.kept == ref.kept == int(B.sum())
    Wh = to_bits(gs.unpack(p))
    assert np.array_equal(Wh, orc.unpack_groups(ref))
    assert np.array_equal(Wh, orc.masked_weight_bits(Wb, B, g, g))


@pytest.mark.parametrize("g", [16, 32, 64, 128])
@pytest.mark.parametrize("T", [1, 3, 8, 9, 16, 17, 32, 33, 48, 64, 128, 129, 300])
def test_linear_small_layers(gs, g, T):
    for out, inp, d, seed in [(256, 512, 0.5, 11), (384, 1024, 0.3, 12), (128, 128, 1.0, 13)]:
        Wb, B, p = make(gs, out, inp, g, d, seed)
        xb = wl.random_activation_bits(T, inp, seed=T + seed)
        y = gs.linear(to_dev(xb), p)
        check_y(to_bits(y), xb, Wb, B, g, what=f"g={g} {out}x{inp} T={T}")


@pytest.mark.parametrize("g", [16, 32])
@pytest.mark.parametrize("T", [1, 40, 300])
def test_linear_input_not_whole_slabs(gs, g, T):
    # in = 3 g is not a multiple of 64 columns: these layers stay on the tile-operand kernel above
    # the decode regime, beside a layer of the same g that takes the zero-filled kernel
    import torch
    layers = [make(gs, 4 * g, 3 * g, g, 0.6, 80 + g), make(gs, 256, 256, g, 0.5, 81 + g)]
    xbs = [wl.random_activation_bits(T, Wb.shape[1], seed=82 + T) for Wb, _, _ in layers]
    ys = [torch.empty((T, Wb.shape[0]), dtype=torch.bfloat16, device="cuda") for Wb, _, _ in layers]
    gs.linear_batched_into([to_dev(b) for b in xbs], [p for _, _, p in layers], ys)
    for (Wb, B, _), xb, y in zip(layers, xbs, ys):
        check_y(to_bits(y), xb, Wb, B, g, what=f"g={g} {Wb.shape} T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("g", [16, 32, 64, 128])
@pytest.mark.parametrize("T", [1, 16, 2048])
def test_linear_llama_block_shapes(gs, g, T):
    # the 7B block's projection shapes at d = 0.5 (token sample above 16)
    for out, inp, seed in [(4096, 4096, 21), (11008, 4096, 22), (4096, 11008, 23)]:
        Wb, B, p = make(gs, out, inp, g, 0.5, seed)
        xb = wl.random_activation_bits(T, inp, seed=T + seed)
        y = to_bits(gs.linear(to_dev(xb), p))
        toks = None if T <= 16 else sample_tokens(T, seed)
        check_y(y, xb, Wb, B, g, tokens=toks, what=f"g={g} {out}x{inp} T={T}")


def test_outliers_zero_rows_and_empty_layers(gs):
    import torch
    g = 32
    # a window whose block rows are all pruned, a layer with nothing kept, x outliers
    out, inp = 512, 1024
    Wb = wl.random_weight_bits(out, inp, seed=31)
    B = wl.random_mask(out // g, inp // g, 0.5, seed=32)
    B[0:4, :] = 0                        # block rows 0..3 = the whole first 128-row window
    B[9, :] = 0                          # one block row pruned everywhere
    p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), g, g)
    p0 = gs.pack_groups(to_dev(Wb), torch.zeros((out // g, inp // g), dtype=torch.uint8, device="cuda"), g, g)
    assert p0.kept == 0
    for T in (5, 40):   # the decode-regime and the tensor-core kernels
        xb = wl.random_activation_bits(T, inp, seed=33)
        xf = wl.bf16_bits_to_f32(xb)
        xf[:, ::97] *= 20.0
        xb = wl.f32_to_bf16_bits(xf)
        y = to_bits(gs.linear(to_dev(xb), p))
        check_y(y, xb, Wb, B, g, what=f"pruned window T={T}")
        assert not y[:, :128].any() and not y[:, 9 * g:10 * g].any()
        y0 = gs.linear(to_dev(xb), p0)
        assert not to_bits(y0).any()


def test_batched_mixes_shapes(gs):
    import torch
    layers = []
    for i, g in enumerate([16, 32, 64, 128, 128, 1]):
        out, inp = (1024, 2048) if g > 1 else (1024, 2048)
        Wb = wl.random_weight_bits(out, inp, seed=40 + i)
        if g == 1:
            B = wl.random_mask(out, inp // 256, 0.5, seed=50 + i)
            p = gs.pack(to_dev(Wb), torch.from_numpy(B).cuda())
            gi = 256
        else:
            B = wl.random_mask(out // g, inp // g, 0.5, seed=50 + i)
            p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), g, g)
            gi = g
        layers.append((Wb, B, p, g, gi))
    for T in (7, 200):
        xbs = [wl.random_activation_bits(T, 2048, seed=60 + i + T) for i in range(len(layers))]
        ys = [torch.empty((T, 1024), dtype=torch.bfloat16, device="cuda") for _ in layers]
        gs.linear_batched_into([to_dev(b) for b in xbs], [l[2] for l in layers], ys)
        for (Wb, B, p, g, gi), xb, y in zip(layers, xbs, ys):
            yr, A = orc.linear(xb, Wb, B, g, gi)
            err = np.abs(bf16_to_f64(to_bits(y)) - yr)
            assert np.all(err <= REL * A + ABS), (g, T)
    assert gs.device_status() == gs.GS_OK


def test_deterministic_and_group_shape_reported(gs):
    Wb, B, p = make(gs, 1024, 1024, 64, 0.5, 70)
    xb = wl.random_activation_bits(256, 1024, seed=71)
    x = to_dev(xb)
    a = to_bits(gs.linear(x, p))
    b = to_bits(gs.linear(x, p))
    assert np.array_equal(a, b)
    import ctypes
    go, gi = ctypes.c_int32(), ctypes.c_int32()
    assert gs.lib.gs_packed_group_shape(p.handle, ctypes.byref(go), ctypes.byref(gi)) == 0
    assert (go.value, gi.value) == (64, 64)


# --------------------------------------------------------------------- 1 x 128 groups

def window_metadata(B):
    """Per (chunk, 16-row window): first packed row and kept-row bitmask, derived
    from the mask by counting (the layout's definition with 128-wide chunks)."""
    out, G = B.shape
    nw = (out + 15) // 16
    win = np.zeros((G, nw + 1), np.int64)
    km = np.zeros((G, nw), np.int64)
    pos = 0
    for c in range(G):
        for w in range(nw):
            win[c, w] = pos
            for i in range(16):
                r = 16 * w + i
                if r < out and B[r, c]:
                    km[c, w] |= 1 << i
                    pos += 1
        win[c, nw] = pos
    return win, km


@pytest.mark.parametrize("out,inp,d,seed", [(1, 128, 1.0, 1), (17, 384, 0.5, 2), (300, 768, 0.5, 3),
                                            (4096, 4096, 0.5, 4), (11008, 4096, 0.45, 5), (4096, 11008, 0.5, 6),
                                            (512, 3584, 0.3, 7), (129, 256, 0.0, 8)])
def test_narrow_rows_pack_and_unpack(gs, out, inp, d, seed):
    import torch
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    B = wl.random_mask(out, inp // 128, d, seed=seed + 900)
    p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), 1, 128)
    ref = orc.pack_groups(Wb, B, 1, 128)
    got = p.export()
    assert np.array_equal(got["offsets"], ref.offsets)
    assert np.array_equal(got["row_idx"], ref.block_row)
    assert np.array_equal(got["tiles"], ref.tiles.reshape(-1, 128))
    win, km = window_metadata(B)
    assert np.array_equal(got["win_off16"], win) and np.array_equal(got["kmask16"], km)
    Wh = to_bits(gs.unpack(p))
    assert np.array_equal(Wh, orc.unpack_groups(ref))


@pytest.mark.parametrize("T", [1, 5, 16, 17, 33, 64, 128, 129, 300, 2048])
def test_narrow_rows_linear(gs, T):
    import torch
    for out, inp, d, seed in [(300, 768, 0.5, 11), (4096, 4096, 0.5, 12), (4096, 11008, 0.5, 13),
                              (512, 3584, 0.3, 14)]:
        Wb = wl.random_weight_bits(out, inp, seed=seed)
        B = wl.random_mask(out, inp // 128, d, seed=seed + 900)
        p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), 1, 128)
        xb = wl.random_activation_bits(T, inp, seed=T + seed)
        x = to_dev(xb)
        toks = None if T <= 300 else sample_tokens(T, seed)
        algos = (gs.ALGO_PREFILL, gs.ALGO_PREFILL_DENSE)
        for algo in ((gs.ALGO_DECODE,) + algos if T <= 300 else algos):
            y = to_bits(gs.linear(x, p, algo=algo))
            if toks is None:
                yr, A = orc.linear(xb, Wb, B, 1, 128)
                yg = bf16_to_f64(y)
            else:
                yr, A = orc.linear_tokens(xb, Wb, B, toks, 1, 128)
                yg = bf16_to_f64(y[np.asarray(toks)])
            assert np.all(np.abs(yg - yr) <= REL * A + ABS), (out, inp, T, algo)


def test_narrow_rows_batched_with_other_shapes(gs):
    import torch
    shapes = [(1, 128), (1, 256), (32, 32), (1, 128)]
    layers = []
    for i, (go, gi) in enumerate(shapes):
        Wb = wl.random_weight_bits(1024, 2048, seed=80 + i)
        B = wl.random_mask(1024 // go, 2048 // gi, 0.5, seed=90 + i)
        p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), go, gi)
        layers.append((Wb, B, p, go, gi))
    # 64 and 200: the 1 x 128 layers take the zero-filled prefill kernel, the 1 x 256 layer the
    # gathering one and the 32 x 32 layer the zero-filled one (above its decode regime)
    for T in (3, 16, 64, 200, 1024):
        xbs = [wl.random_activation_bits(T, 2048, seed=100 + i + T) for i in range(len(layers))]
        ys = [torch.empty((T, 1024), dtype=torch.bfloat16, device="cuda") for _ in layers]
        gs.linear_batched_into([to_dev(b) for b in xbs], [l[2] for l in layers], ys)
        for (Wb, B, p, go, gi), xb, y in zip(layers, xbs, ys):
            yr, A = orc.linear(xb, Wb, B, go, gi)
            assert np.all(np.abs(bf16_to_f64(to_bits(y)) - yr) <= REL * A + ABS), (go, gi, T)
            # a batched call gives each layer what a single call gives it, bit for bit
            assert np.array_equal(to_bits(y), to_bits(gs.linear(to_dev(xb), p))), (go, gi, T)
    assert gs.device_status() == gs.GS_OK
