"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each test targets a plausible mistake: a dropped or extra group, a wrong sign,
a transposed operand or mask, a wrong group orientation, a wrong packing order.
Sources of truth: hand-derived golden fixtures (tests/golden), exact integer
arithmetic (Python / numpy int64), correctly rounded sums (math.fsum), brute
force over every mask of tiny layers, and identities that Eq. 1 implies
(complement, disjoint union, permutation equivariance, scaling).
"""
import itertools
import json
import math
from pathlib import Path

import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl

GOLDEN = Path(__file__).resolve().parent / "golden"


def bits_of(a):
    return wl.f32_to_bf16_bits(np.asarray(a, dtype=np.float32))


def const_groups(vals, width=256):
    """Expand a [rows, G] table of constants into a [rows, G*width] bf16 bit matrix."""
    v = np.repeat(np.asarray(vals, dtype=np.float32), width, axis=1)
    return bits_of(v)


def int_bits(rng, shape, lo=-4, hi=4):
    """bf16 bits of small integers (exact in bf16), and the integers."""
    ints = rng.integers(lo, hi + 1, size=shape)
    return bits_of(ints.astype(np.float32)), ints.astype(np.int64)


def int_reference(x_int, W_int, B):
    """Exact y via int64 arithmetic, summing kept groups chunk by chunk."""
    T = x_int.shape[0]
    out, G = B.shape
    y = np.zeros((T, out), dtype=np.int64)
    for r in range(out):
        for c in range(G):
            if B[r, c]:
                y[:, r] += x_int[:, 256 * c:256 * (c + 1)] @ W_int[r, 256 * c:256 * (c + 1)]
    return y


# --------------------------------------------------------------------- golden

def test_golden_tiny_layer():
    g = json.loads((GOLDEN / "tiny_layer.json").read_text())
    B = np.asarray(g["mask"], dtype=np.uint8)
    W = const_groups(g["W_const"])
    x = const_groups(g["x_const"])
    assert W.shape == (g["out"], g["in"])
    y, A = orc.linear(x, W, B)
    e = g["expected"]
    assert np.array_equal(y, np.asarray(e["y"]))
    assert np.array_equal(A, np.asarray(e["A"]))
    p = orc.pack(W, B)
    assert p.offsets.tolist() == e["offsets"]
    assert p.row_idx.tolist() == e["row_idx"]
    assert np.array_equal(p.tiles, const_groups(np.asarray(e["tile_const"])[:, None]))
    assert p.kmask16.tolist() == e["kmask16"]
    assert p.win_off16.tolist() == e["win_off16"]
    assert orc.layer_sparsity(B) == pytest.approx(e["layer_sparsity"], abs=0, rel=1e-15)


def test_golden_global_sparsity():
    g = json.loads((GOLDEN / "global_sparsity.json").read_text())
    Bs = [np.asarray(l["mask"]) for l in g["layers"]]
    shapes = [(l["d_out"], l["d_in"]) for l in g["layers"]]
    for B, l in zip(Bs, g["layers"]):
        assert orc.layer_sparsity(B) == l["s"]
    assert orc.global_sparsity(Bs, shapes) == g["s_global"]


# --------------------------------------------------------------------- exact integer cases

@pytest.mark.parametrize("seed", [0, 1, 2])
def test_exact_integer_layer(seed):
    rng = np.random.default_rng(seed)
    out, inp, T = 5, 768, 3
    xb, xi = int_bits(rng, (T, inp))
    Wb, Wi = int_bits(rng, (out, inp))
    B = (rng.random((out, inp // 256)) < 0.5).astype(np.uint8)
    y, A = orc.linear(xb, Wb, B)
    yi = int_reference(xi, Wi, B)
    assert np.array_equal(y, yi.astype(np.float64))
    Ai = int_reference(np.abs(xi), np.abs(Wi), B)
    assert np.array_equal(A, Ai.astype(np.float64))


def test_brute_force_every_mask_tiny():
    rng = np.random.default_rng(7)
    out, inp, T = 2, 512, 2
    xb, xi = int_bits(rng, (T, inp), -8, 8)
    Wb, Wi = int_bits(rng, (out, inp), -8, 8)
    G = inp // 256
    for bits in itertools.product([0, 1], repeat=out * G):
        B = np.asarray(bits, dtype=np.uint8).reshape(out, G)
        y, _ = orc.linear(xb, Wb, B)
        assert np.array_equal(y, int_reference(xi, Wi, B).astype(np.float64)), bits


def test_all_kept_is_dense_product_and_all_pruned_is_zero():
    rng = np.random.default_rng(3)
    out, inp, T = 4, 1024, 3
    xb, xi = int_bits(rng, (T, inp))
    Wb, Wi = int_bits(rng, (out, inp))
    ones = np.ones((out, inp // 256), np.uint8)
    y, _ = orc.linear(xb, Wb, ones)
    assert np.array_equal(y, (xi @ Wi.T).astype(np.float64))      # B = 1: the dense teacher
    y0, A0 = orc.linear(xb, Wb, np.zeros_like(ones))
    assert not np.any(y0) and not np.any(A0)


def test_complement_and_disjoint_union():
    rng = np.random.default_rng(4)
    out, inp, T = 6, 1280, 2
    xb, _ = int_bits(rng, (T, inp))
    Wb, _ = int_bits(rng, (out, inp))
    G = inp // 256
    B1 = (rng.random((out, G)) < 0.3).astype(np.uint8)
    B2 = ((rng.random((out, G)) < 0.5) & (B1 == 0)).astype(np.uint8)
    y1, _ = orc.linear(xb, Wb, B1)
    y2, _ = orc.linear(xb, Wb, B2)
    y12, _ = orc.linear(xb, Wb, B1 | B2)
    yc, _ = orc.linear(xb, Wb, 1 - B1)
    yd, _ = orc.linear(xb, Wb, np.ones_like(B1))
    assert np.array_equal(y1 + y2, y12)
    assert np.array_equal(y1 + yc, yd)


def test_one_hot_group_orientation():
    """Keeping a single group (r0, c0) must touch only output r0 and only input
    columns 256*c0 .. 256*c0+255 (groups run along the input dimension)."""
    rng = np.random.default_rng(5)
    out, inp, T = 3, 768, 2
    xb = wl.random_activation_bits(T, inp, seed=11)
    Wb = wl.random_weight_bits(out, inp, seed=12)
    x = wl.bf16_bits_to_f64(xb)
    W = wl.bf16_bits_to_f64(Wb)
    for r0 in range(out):
        for c0 in range(inp // 256):
            B = np.zeros((out, inp // 256), np.uint8)
            B[r0, c0] = 1
            y, _ = orc.linear(xb, Wb, B)
            for t in range(T):
                for r in range(out):
                    if r != r0:
                        assert y[t, r] == 0.0
                ref = math.fsum(x[t, 256 * c0 + k] * W[r0, 256 * c0 + k] for k in range(256))
                assert y[t, r0] == pytest.approx(ref, rel=1e-13, abs=1e-300)


def test_against_correctly_rounded_sums():
    out, inp, T = 4, 768, 3
    xb = wl.random_activation_bits(T, inp, seed=21)
    Wb = wl.random_weight_bits(out, inp, seed=22)
    B = wl.random_mask(out, inp // 256, 0.6, seed=23)
    x = wl.bf16_bits_to_f64(xb)
    W = wl.bf16_bits_to_f64(Wb)
    y, A = orc.linear(xb, Wb, B)
    for t in range(T):
        for r in range(out):
            terms = [x[t, 256 * c + k] * W[r, 256 * c + k]
                     for c in range(inp // 256) if B[r, c] for k in range(256)]
            ref = math.fsum(terms)
            aref = math.fsum(abs(v) for v in terms)
            assert abs(y[t, r] - ref) <= 1e-14 * aref + 1e-300
            assert A[t, r] == pytest.approx(aref, rel=1e-14, abs=0)
            assert abs(y[t, r]) <= A[t, r]


def test_permutation_equivariance_and_scaling():
    rng = np.random.default_rng(6)
    out, inp, T = 5, 1024, 3
    xb, _ = int_bits(rng, (T, inp))
    Wb, _ = int_bits(rng, (out, inp))
    G = inp // 256
    B = (rng.random((out, G)) < 0.5).astype(np.uint8)
    y, _ = orc.linear(xb, Wb, B)
    # permuting output rows (W rows and mask rows) permutes y's columns
    pr = rng.permutation(out)
    yp, _ = orc.linear(xb, Wb[pr], B[pr])
    assert np.array_equal(yp, y[:, pr])
    # permuting whole 256-wide chunks of x, W and the mask columns leaves y unchanged
    pc = rng.permutation(G)
    cols = np.concatenate([np.arange(256 * c, 256 * (c + 1)) for c in pc])
    yc, _ = orc.linear(xb[:, cols], Wb[:, cols], B[:, pc])
    assert np.array_equal(yc, y)
    # permuting tokens permutes y's rows; scaling x by 2 scales y by 2 (exact in binary)
    pt = rng.permutation(T)
    yt, _ = orc.linear(xb[pt], Wb, B)
    assert np.array_equal(yt, y[pt])
    x2 = bits_of(wl.bf16_bits_to_f32(xb) * np.float32(2.0))
    y2, _ = orc.linear(x2, Wb, B)
    assert np.array_equal(y2, 2.0 * y)


# --------------------------------------------------------------------- packing

@pytest.mark.parametrize("out,inp,d,seed", [(1, 256, 1.0, 0), (17, 512, 0.5, 1), (40, 1280, 0.3, 2),
                                             (33, 768, 0.0, 3), (64, 256, 1.0, 4)])
def test_pack_invariants_and_roundtrip(out, inp, d, seed):
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    B = wl.random_mask(out, inp // 256, d, seed=seed + 100)
    p = orc.pack(Wb, B)
    G = inp // 256
    assert p.offsets[0] == 0 and p.kept == int(B.sum())
    assert np.all(np.diff(p.offsets) == B.sum(axis=0))               # n_c = #kept rows of chunk c
    for c in range(G):
        rows = p.row_idx[p.offsets[c]:p.offsets[c + 1]]
        assert np.all(np.diff(rows) > 0)                              # ascending, distinct
        assert all(B[r, c] for r in rows)
        for j, r in zip(range(p.offsets[c], p.offsets[c + 1]), rows):
            assert np.array_equal(p.tiles[j], Wb[r, 256 * c:256 * (c + 1)])
    # window metadata: brute force from the mask
    nw16 = (out + 15) // 16
    for c in range(G):
        for w in range(nw16):
            rows = [r for r in range(16 * w, min(16 * w + 16, out)) if B[r, c]]
            assert p.kmask16[c, w] == sum(1 << (r - 16 * w) for r in rows)
            assert p.win_off16[c, w] == p.offsets[c] + int(B[:16 * w, c].sum())
        assert p.win_off16[c, nw16] == p.offsets[c + 1]
    # unpack reproduces W (.) M bit-exactly, pruned = +0.0
    assert np.array_equal(orc.unpack(p), orc.masked_weight_bits(Wb, B))


def test_masked_weight_uses_positive_zero():
    Wb = bits_of(-np.ones((2, 512), np.float32))
    B = np.array([[1, 0], [0, 1]], np.uint8)
    Wh = orc.masked_weight_bits(Wb, B)
    assert np.all(Wh[0, 256:] == 0) and np.all(Wh[1, :256] == 0)
    assert np.all(Wh[0, :256] == 0xBF80) and np.all(Wh[1, 256:] == 0xBF80)
    assert np.all(np.signbit(orc.masked_weight(Wb, B)) == (Wh == 0xBF80))


def test_packed_route_equals_definition():
    out, inp, T = 6, 768, 2
    xb = wl.random_activation_bits(T, inp, seed=31)
    Wb = wl.random_weight_bits(out, inp, seed=32)
    B = wl.random_mask(out, inp // 256, 0.5, seed=33)
    y, A = orc.linear(xb, Wb, B)
    yp = orc.linear_packed(xb, orc.pack(Wb, B))
    assert np.all(np.abs(yp - y) <= 1e-14 * A + 1e-300)


# --------------------------------------------------------------------- Eq. 2 / App. F

def test_sparsity_closed_forms():
    assert orc.layer_sparsity(np.ones((4, 3))) == 0.0
    assert orc.layer_sparsity(np.zeros((4, 3))) == 1.0
    B = np.zeros((8, 4), np.uint8)
    B[:, :2] = 1
    assert orc.layer_sparsity(B) == 0.5
    # with 1x256 groups every group holds 256 weights: preserved rate = 1 - s^l
    rng = np.random.default_rng(0)
    B = (rng.random((10, 6)) < 0.37).astype(np.uint8)
    assert orc.preserved_rate(B) == pytest.approx(1.0 - orc.layer_sparsity(B), abs=1e-15)
    # square groups (g_out = g_in = 2): each selector covers 4 weights
    Bs = np.array([[1, 0], [0, 0]])
    assert orc.expand_mask(Bs, 2, 2).sum() == 4 and orc.expand_mask(Bs, 2, 2)[:2, :2].all()


def test_bf16_rounding_helper():
    # round-to-nearest-even on hand-picked values
    v = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -7, -2.5, 0.0], np.float32)
    assert wl.f32_to_bf16_bits(v).tolist() == [0x3F80, 0x3F80, 0x3F82, 0x3F81, 0xC020, 0x0000]
    assert np.array_equal(wl.bf16_bits_to_f32(np.array([0x3F80, 0xC020], np.uint16)), np.array([1.0, -2.5], np.float32))


# --------------------------------------------------------------------- Sec. 2.2 / App. F: selector export

def test_golden_selector_threshold():
    g = json.loads((GOLDEN / "selector_threshold.json").read_text())
    raw = np.array([int(h, 16) for h in g["logits_hex_f32"]], dtype=np.uint32).view(np.float32)
    assert orc.select_groups(raw).tolist() == g["selector"]
    assert orc.select_groups(raw).dtype == np.uint8


@pytest.mark.parametrize("tau", [0.25, 1.0, 4.0])
def test_selector_matches_sigmoid_away_from_zero(tau):
    special = pytest.importorskip("scipy.special")
    rng = np.random.default_rng(7)
    lg = (rng.standard_normal((64, 37)) * 3.0).astype(np.float32)
    lg[np.abs(lg) < 1e-6] = 1.0
    # the noise-free Gumbel-Sigmoid relaxation at any temperature, thresholded at 1/2
    ref = (special.expit(lg.astype(np.float64) / tau) > 0.5).astype(np.uint8)
    assert np.array_equal(orc.select_groups(lg), ref)


def test_selector_sign_symmetry_and_shape():
    rng = np.random.default_rng(8)
    lg = rng.standard_normal((5, 9)).astype(np.float32)
    B = orc.select_groups(lg)
    assert B.shape == (5, 9)
    assert np.array_equal(orc.select_groups(-lg), 1 - B)          # no zeros among these logits
    assert orc.kept_groups(B) == int(np.count_nonzero(lg > 0))


def test_global_preserved_rate_reproduces_the_printed_allocation():
    g = json.loads((GOLDEN / "llama2_7b_allocation.json").read_text())
    Bs, shapes = [], []
    for name, (d_out, d_in) in g["shapes"].items():
        rate = g["attention_rate"] if name in ("q", "k", "v", "o") else g["mlp_rate"]
        n = d_out * d_in // 256
        B = np.zeros((d_out, d_in // 256), np.uint8)
        B.reshape(-1)[: int(round(rate * n))] = 1
        Bs.append(B)
        shapes.append((d_out, d_in))
    got = orc.global_preserved_rate(Bs, shapes)
    tol = g["printed_rate_half_unit"] + g["global_half_unit"] + 1e-6
    assert abs(got - g["global_preserved"]) <= tol
    # an unweighted mean over the projections misses the printed figure by far
    unweighted = float(np.mean([orc.preserved_rate(B) for B in Bs]))
    assert abs(unweighted - g["global_preserved"]) > 10 * tol


def test_global_preserved_rate_is_one_minus_golden_sparsity():
    g = json.loads((GOLDEN / "global_sparsity.json").read_text())
    Bs = [np.asarray(l["mask"]) for l in g["layers"]]
    shapes = [(l["d_out"], l["d_in"]) for l in g["layers"]]
    assert orc.global_preserved_rate(Bs, shapes) == 1.0 - g["s_global"]


def test_qkv_rate_is_the_plain_mean():
    # q keeps its only group, k keeps 2 of 8, v keeps none: (1 + 0.25 + 0) / 3
    Bq = np.ones((1, 1), np.uint8)
    Bk = np.zeros((4, 2), np.uint8)
    Bk[0, 0] = Bk[3, 1] = 1
    Bv = np.zeros((2, 1), np.uint8)
    assert orc.qkv_preserved_rate(Bq, Bk, Bv) == pytest.approx(1.25 / 3, abs=1e-15)
    # a parameter-weighted mean would give (256 + 512) / (256 + 2048 + 512)
    assert abs(orc.qkv_preserved_rate(Bq, Bk, Bv) - 768 / 2816) > 0.1


# --------------------------------------------------------------------- other group shapes (Sec. 2.1, Sec. 3.5, App. E)

@pytest.mark.parametrize("g", [16, 32])
def test_one_hot_square_group_orientation(g):
    # a single kept g x g group (u, v) of a 2g x 3g weight keeps exactly rows g*u..g*u+g-1
    # and columns g*v..g*v+g-1 (checked cell by cell, no Kronecker product)
    vals = np.arange(1, 2 * g * 3 * g + 1, dtype=np.float32).reshape(2 * g, 3 * g) % 200 + 1
    Wb = bits_of(vals)
    for u in range(2):
        for v in range(3):
            B = np.zeros((2, 3), np.uint8)
            B[u, v] = 1
            got = orc.masked_weight_bits(Wb, B, g, g)
            for r in range(2 * g):
                for k in range(3 * g):
                    inside = (g * u <= r < g * u + g) and (g * v <= k < g * v + g)
                    assert got[r, k] == (Wb[r, k] if inside else 0)


def test_brute_force_every_square_mask_tiny():
    # 32 x 32 weight, 16 x 16 groups: all 16 masks; y by int64 loops where group
    # membership is the integer division B[r // 16, k // 16]
    rng = np.random.default_rng(11)
    Wb, Wi = int_bits(rng, (32, 32))
    xb, xi = int_bits(rng, (3, 32))
    for bits in range(16):
        B = np.array([[(bits >> 0) & 1, (bits >> 1) & 1], [(bits >> 2) & 1, (bits >> 3) & 1]], np.uint8)
        ref = np.zeros((3, 32), np.int64)
        for t in range(3):
            for r in range(32):
                ref[t, r] = sum(int(xi[t, k]) * int(Wi[r, k]) for k in range(32) if B[r // 16, k // 16])
        y, _ = orc.linear(xb, Wb, B, 16, 16)
        assert np.array_equal(y, ref.astype(np.float64)), bits
        assert np.array_equal(orc.linear_packed_groups(xb, orc.pack_groups(Wb, B, 16, 16)), ref.astype(np.float64))


def test_square_and_narrow_masks_reduce_to_row_masks():
    rng = np.random.default_rng(12)
    Wb = wl.random_weight_bits(128, 512, seed=12)
    xb = wl.random_activation_bits(4, 512, seed=13)
    # a 32 x 32 mask is the 1 x 32 mask with each group row repeated 32 times
    Bsq = (rng.random((4, 16)) < 0.5).astype(np.uint8)
    Brow = np.repeat(Bsq, 32, axis=0)
    assert np.array_equal(orc.masked_weight_bits(Wb, Bsq, 32, 32), orc.masked_weight_bits(Wb, Brow, 1, 32))
    y1, _ = orc.linear(xb, Wb, Bsq, 32, 32)
    y2, _ = orc.linear(xb, Wb, Brow, 1, 32)
    assert np.array_equal(y1, y2)
    # a 1 x 128 mask whose column pairs agree is the 1 x 256 mask
    B256 = (rng.random((128, 2)) < 0.5).astype(np.uint8)
    B128 = np.repeat(B256, 2, axis=1)
    assert np.array_equal(orc.masked_weight_bits(Wb, B128, 1, 128), orc.masked_weight_bits(Wb, B256))


def test_pack_groups_reduces_to_the_1x256_layout():
    Wb = wl.random_weight_bits(40, 768, seed=14)
    B = wl.random_mask(40, 3, 0.5, seed=15)
    pg, p = orc.pack_groups(Wb, B, 1, 256), orc.pack(Wb, B)
    assert np.array_equal(pg.offsets, p.offsets) and np.array_equal(pg.block_row, p.row_idx)
    assert np.array_equal(pg.tiles.reshape(-1, 256), p.tiles)


@pytest.mark.parametrize("g_out,g_in", orc.GROUP_SHAPES)
def test_pack_groups_roundtrip_counts_and_route(g_out, g_in):
    out, inp = 256, 512
    Wb = wl.random_weight_bits(out, inp, seed=16)
    xb = wl.random_activation_bits(3, inp, seed=17)
    Go, Gi = orc.group_grid(out, inp, g_out, g_in)
    B = (np.random.default_rng(g_out * 1000 + g_in).random((Go, Gi)) < 0.45).astype(np.uint8)
    p = orc.pack_groups(Wb, B, g_out, g_in)
    assert p.kept == int(B.sum()) and p.tiles.shape == (p.kept, g_out, g_in)
    assert np.all(np.diff(p.offsets) >= 0)
    for v in range(Gi):
        rows = p.block_row[p.offsets[v]:p.offsets[v + 1]]
        assert rows.tolist() == [u for u in range(Go) if B[u, v]]
    assert np.array_equal(orc.unpack_groups(p), orc.masked_weight_bits(Wb, B, g_out, g_in))
    y, A = orc.linear(xb, Wb, B, g_out, g_in)
    assert np.all(np.abs(orc.linear_packed_groups(xb, p) - y) <= 1e-13 * A + 1e-300)
    assert orc.preserved_rate(B, g_out, g_in) == p.kept * g_out * g_in / (out * inp)


def test_group_grid_rejects_untiled_shapes():
    assert orc.group_grid(11008, 4096, 128, 128) == (86, 32)
    with pytest.raises(ValueError):
        orc.group_grid(100, 256, 16, 16)
    with pytest.raises(ValueError):
        orc.group_grid(128, 200, 1, 128)


def test_golden_square_layout():
    g = json.loads((GOLDEN / "square_layout.json").read_text())
    W = bits_of(np.asarray(g["W"], np.float32))
    B = np.asarray(g["mask"], np.uint8)
    x = bits_of(np.asarray(g["x"], np.float32))
    e = g["expected"]
    p = orc.pack_groups(W, B, g["g"], g["g"])
    assert p.offsets.tolist() == e["offsets"] and p.block_row.tolist() == e["block_row"]
    assert np.array_equal(p.tiles, bits_of(np.asarray(e["tiles"], np.float32)))
    y, _ = orc.linear(x, W, B, g["g"], g["g"])
    assert np.array_equal(y, np.asarray(e["y"], np.float64))
    assert np.array_equal(orc.linear_packed_groups(x, p), np.asarray(e["y"], np.float64))
    assert orc.preserved_rate(B, g["g"], g["g"]) == e["preserved_rate"]


# --------------------------------------------------------------------- token subsets and kept counts

def test_golden_token_rows():
    # linear_tokens returns the listed rows, in the listed order, repeats included
    g = json.loads((GOLDEN / "token_rows.json").read_text())
    B = np.asarray(g["mask"], dtype=np.uint8)
    W = const_groups(g["W_const"])
    x = const_groups(g["x_const"])
    y, A = orc.linear_tokens(x, W, B, g["tokens"])
    e = g["expected"]
    assert np.array_equal(y, np.asarray(e["y"]))
    assert np.array_equal(A, np.asarray(e["A"]))
    assert orc.kept_groups(B) == e["kept_groups"]


@pytest.mark.parametrize("seed", [0, 1])
def test_token_rows_against_integer_loops(seed):
    # every listed token row equals the exact int64 layer output of that token;
    # the list is unsorted and repeats entries (a sorted or deduplicated result fails)
    rng = np.random.default_rng(100 + seed)
    out, inp, T = 7, 1024, 6
    xb, xi = int_bits(rng, (T, inp))
    Wb, Wi = int_bits(rng, (out, inp))
    B = (rng.random((out, inp // 256)) < 0.5).astype(np.uint8)
    tokens = [5, 1, 1, 3, 0, 5]
    y, A = orc.linear_tokens(xb, Wb, B, tokens)
    assert y.shape == (len(tokens), out)
    for i, t in enumerate(tokens):
        assert np.array_equal(y[i], int_reference(xi[t:t + 1], Wi, B)[0].astype(np.float64))
        assert np.array_equal(A[i], int_reference(np.abs(xi[t:t + 1]), np.abs(Wi), B)[0].astype(np.float64))


def test_kept_groups_counts_nonzero_bytes_as_keep():
    # mask bytes are keep-if-nonzero: 3, 255 and 1 all keep; the count is the
    # numerator of Eq. 2, here written out by hand
    B = np.array([[0, 3, 0, 0], [255, 0, 0, 1], [1, 1, 0, 0]], dtype=np.uint8)
    assert orc.kept_groups(B) == 5
    assert orc.kept_groups(np.zeros((9, 4), np.uint8)) == 0
    assert orc.kept_groups(np.ones((9, 4), np.uint8)) == 36
    assert orc.kept_groups(B.astype(bool)) == 5


def test_kept_groups_matches_the_allocated_budget():
    # the seeded generator places exactly k_l groups per layer (its own top-k
    # recipe, no oracle code); the oracle's count must return each k_l and the sum
    from paper_2609_33977_gb300 import workload as wl_mod
    w = wl_mod.workload(2)
    ks = wl_mod.keep_counts(w)
    total = 0
    for i in (0, 4, 6):
        B = wl_mod.group_mask(w, i, int(ks[i]))
        assert orc.kept_groups(B) == int(ks[i])
        total += orc.kept_groups(B)
    assert total == int(ks[0] + ks[4] + ks[6])


# --------------------------------------------------------------------- Gumbel-Sigmoid + straight-through (Sec. 2.2)

def test_golden_gumbel_select():
    g = json.loads((GOLDEN / "gumbel_select.json").read_text())
    B, s = orc.gumbel_select(np.asarray(g["logits"], np.float32), np.asarray(g["noise"], np.float32), g["tau"])
    e = g["expected"]
    assert B.tolist() == e["mask"]
    for i, v in enumerate(e["sum"]):
        if v == 0.0:
            assert s[i] == e["soft_at_zero"]
    for case in g["ln3_cases"]:
        tau = abs(case["logit"] + case["noise"]) / math.log(3.0)
        Bc, sc = orc.gumbel_select(np.float32([case["logit"]]), np.float32([case["noise"]]), tau)
        assert int(Bc[0]) == case["mask"]
        assert sc[0] == pytest.approx(case["soft"], abs=1e-15)


@pytest.mark.parametrize("tau", [0.4, 1.0, 2.5])
def test_gumbel_select_matches_library_sigmoid_and_threshold(tau):
    from scipy.special import expit
    rng = np.random.default_rng(5)
    lg = rng.standard_normal(4000).astype(np.float32)
    u = rng.random(4000)
    noise = (np.log(u) - np.log1p(-u)).astype(np.float32)     # logistic = difference of two Gumbels
    B, s = orc.gumbel_select(lg, noise, tau)
    z = (lg + noise).astype(np.float64)
    assert np.allclose(s, expit(z / tau), rtol=1e-14, atol=0)
    assert np.array_equal(B, (z > 0).astype(np.uint8))
    assert np.array_equal(B, (s > 0.5).astype(np.uint8))      # the threshold the paper describes
    # without noise the sample is the evaluation-time export
    assert np.array_equal(orc.gumbel_select(lg, np.zeros_like(lg), tau)[0], orc.select_groups(lg))


def _relaxed_loss(x, W, lg, noise, tau, dy, g_in):
    """sum(dy * y) with y = x (W (.) (s kron 1))^T, s = sigmoid((l + L)/tau): the
    relaxed forward the straight-through backward differentiates (numpy, fp64)."""
    s = 1.0 / (1.0 + np.exp(-(lg + noise) / tau))
    M = np.repeat(s, g_in, axis=1)
    return float(np.sum(dy * (x @ (W * M).T)))


def test_straight_through_backward_against_finite_differences():
    rng = np.random.default_rng(21)
    out, inp, T, tau = 3, 512, 4, 0.4
    xi = rng.integers(-3, 4, size=(T, inp))
    Wi = rng.integers(-3, 4, size=(out, inp))
    xb, Wb = bits_of(xi.astype(np.float32)), bits_of(Wi.astype(np.float32))
    lg = (rng.integers(-8, 9, size=(out, inp // 256)) / 8.0).astype(np.float32)
    noise = (rng.integers(-8, 9, size=lg.shape) / 8.0).astype(np.float32)
    dy = rng.standard_normal((T, out))
    B, s = orc.gumbel_select(lg, noise, tau)
    dl, dx = orc.masked_linear_backward(xb, Wb, B, dy, orc.gumbel_dsdl(lg, noise, tau))
    x, W = xi.astype(np.float64), Wi.astype(np.float64)
    h = 1e-6
    for r in range(out):
        for c in range(inp // 256):
            lp, lm = lg.astype(np.float64), lg.astype(np.float64)
            lp = lp.copy()
            lm = lm.copy()
            lp[r, c] += h
            lm[r, c] -= h
            fd = (_relaxed_loss(x, W, lp, noise.astype(np.float64), tau, dy, 256)
                  - _relaxed_loss(x, W, lm, noise.astype(np.float64), tau, dy, 256)) / (2 * h)
            assert dl[r, c] == pytest.approx(fd, rel=1e-6, abs=1e-6), (r, c)
    # the input gradient uses the binary mask of the forward pass: exact in integers
    Mi = np.repeat(B.astype(np.int64), 256, axis=1)
    dyi = rng.integers(-3, 4, size=(T, out))
    _, dx_int = orc.masked_linear_backward(xb, Wb, B, dyi.astype(np.float64), orc.gumbel_dsdl(lg, noise, tau))
    assert np.array_equal(dx_int, (dyi @ (Wi * Mi)).astype(np.float64))


def test_group_weight_grad_exact_and_oriented():
    # dL/dB[r, c] = sum_k W[r, 256c+k] sum_t dy[t, r] x[t, 256c+k], checked by int64 loops
    rng = np.random.default_rng(22)
    out, inp, T = 5, 768, 3
    xi = rng.integers(-4, 5, size=(T, inp))
    Wi = rng.integers(-4, 5, size=(out, inp))
    dyi = rng.integers(-4, 5, size=(T, out))
    G = orc.group_weight_grad(bits_of(xi.astype(np.float32)), bits_of(Wi.astype(np.float32)), dyi.astype(np.float64))
    assert G.shape == (out, inp // 256)
    for r in range(out):
        for c in range(inp // 256):
            ref = 0
            for k in range(256 * c, 256 * c + 256):
                ref += int(Wi[r, k]) * int(sum(int(dyi[t, r]) * int(xi[t, k]) for t in range(T)))
            assert G[r, c] == float(ref)
    # square groups: the 16x16 group sums reduce the same cell products
    Gs = orc.group_weight_grad(bits_of(xi[:, :256].astype(np.float32)),
                               bits_of(np.tile(Wi[:1, :256], (16, 1)).astype(np.float32)),
                               np.tile(dyi[:, :1], (1, 16)).astype(np.float64), 16, 16)
    assert Gs.shape == (1, 16)
    cell = np.tile(Wi[:1, :256], (16, 1)) * (np.tile(dyi[:, :1], (1, 16)).T @ xi[:, :256])
    assert np.array_equal(Gs, cell.reshape(1, 16, 16, 16).sum(axis=(1, 3)).astype(np.float64))


@pytest.mark.parametrize("tau", [0.4, 1.0, 3.0])
def test_gumbel_dsdl_is_the_sigmoid_derivative(tau):
    from scipy.special import expit
    rng = np.random.default_rng(31)
    lg = (rng.standard_normal(2000) * 4).astype(np.float32)
    noise = rng.standard_normal(2000).astype(np.float32)
    d = orc.gumbel_dsdl(lg, noise, tau)
    z = (lg + noise).astype(np.float64)
    # central finite difference of sigmoid(z / tau) in z, taken on the lower
    # tail (sigmoid(-a) for z > 0) where the two values do not cancel
    h = 1e-5
    fd = np.where(z > 0, expit(-(z - h) / tau) - expit(-(z + h) / tau),
                  expit((z + h) / tau) - expit((z - h) / tau)) / (2 * h)
    assert np.allclose(d, fd, rtol=1e-6, atol=1e-12)
    # closed forms: 1 / (4 tau) at z = 0, symmetric in z, and s (1 - s) / tau where that has no cancellation
    assert orc.gumbel_dsdl(np.float32([0.0]), np.float32([0.0]), tau)[0] == 0.25 / tau
    assert np.array_equal(d, orc.gumbel_dsdl(-lg, -noise, tau))
    s = expit(z / tau)
    mid = np.abs(z / tau) < 5
    assert np.allclose(d[mid], (s * (1 - s) / tau)[mid], rtol=1e-12)
    # far in the tails it keeps its relative precision (1 - s would have cancelled)
    far = orc.gumbel_dsdl(np.float32([20.0]), np.float32([0.0]), 0.5)[0]
    assert far == pytest.approx(math.exp(-40.0) / (1 + math.exp(-40.0)) ** 2 / 0.5, rel=1e-14)
