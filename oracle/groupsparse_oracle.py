"""CPU oracle for the group-sparse linear layer  y = x (W (.) M)^T.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import or call
this module: only the test-suite, the package smoke check and the benchmark's
CPU-baseline / reference leg use it.  It shares no code with the CUDA library
and imports nothing from it.

Everything is plain numpy in float64 on the exact bf16 values (bf16 widens to
float64 without rounding).  Each function follows one definition:

* group partition and mask expansion, Sec. 2.1 and Eq. 1:
  M = B (x) 1_{g_out x g_in},  W_hat = W (.) M
* sparsity accounting, Eq. 2: s^l = 1 - sum(B^l) / (G_out G_in),
  s = sum_l s^l d_out d_in / sum_l d_out d_in
* the layer output: y = x W_hat^T (the linear projection the masked weight
  replaces; no bias), computed as one float64 matrix product
* the packed layout (chunk-major kept-row lists, weight tiles, offsets), which
  the paper leaves unspecified; the layout is defined by the sequential loop in
  `pack` below.
* other group shapes, Sec. 2.1 with g_out x g_in groups (1x128 and the square
  16..128 shapes of the Sec. 3.5 ablation and App. E): `linear` takes the
  shape, and `pack_groups` / `unpack_groups` / `linear_packed_groups` define a
  column-major block layout that reduces to `pack`'s for 1x256;
* selector export, Sec. 2.2 and App. F: with the Gumbel noise removed, a
  selector logit l keeps its group when sigmoid(l) > 1/2; App. F applies the
  same rule when the masks are exported, then reports each projection's
  preserved rate (active / total weights), the Q/K/V rates averaged.
* training-side selectors, Sec. 2.2: a Gumbel-Sigmoid sample (logistic noise
  passed in, temperature tau) gives binary selectors for the forward pass and
  a relaxation whose derivative the straight-through estimator uses in the
  backward pass; the backward of y = x W_hat^T gives the selector-logit and
  input gradients.

Readings where the paper is silent (all listed in the design notes):
* groups are 1 x 256 along the input dimension, aligned at multiples of 256;
* M acts as a select, so a pruned weight is +0.0 (bit pattern 0x0000) even
  where W is negative;
* a nonzero mask byte means "keep";
* the export threshold is 1/2 on sigmoid(l), strict (the paper names no
  value): l = +0, l = -0 and NaN logits prune.

Parity pins: every function here is pinned by the `-m "not gpu"` tests in
tests/test_oracle_pins.py (exact integer cases, complement and disjoint-union
identities, one-hot masks, permutation equivariance, hand-derived golden
layouts, closed-form sparsities; for the selector export: hand-derived
threshold cases over the float32 special values, agreement with a library
sigmoid at several temperatures, and the global preserved rate the paper
prints for its LLaMA-2-7B allocation in Sec. 3.5; for other group shapes:
cell-by-cell one-hot orientation, brute force over every 16x16 mask of a
32x32 weight against int64 loops, reduction of square and 1x128 masks to row
masks, and the 1x256 layout identity; for token subsets: a hand-derived golden
case whose token list is out of order and repeats a row, and int64 loops per
listed token; for the kept count: hand-written masks with keep bytes other
than 1, and the exact per-layer budget of the seeded generator; for the
Gumbel-Sigmoid sample: hand-derived decisions and relaxation values, and
agreement with a library sigmoid; for the straight-through backward: central
finite differences of the relaxed forward loss, and exact integer cases).
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Iterable, List, Sequence, Tuple

import numpy as np

G_IN = 256
WIN16 = 16   # row-window height of the per-(chunk, window) metadata in the packed layout


def _bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------------------
# Eq. 1: mask expansion and masked weight
# ---------------------------------------------------------------------------

def expand_mask(B: np.ndarray, g_out: int = 1, g_in: int = G_IN) -> np.ndarray:
    """M = B (x) 1_{g_out x g_in} (Kronecker product, Eq. 1) as a boolean matrix."""
    B = (np.asarray(B) != 0).astype(np.uint8)
    return np.kron(B, np.ones((g_out, g_in), dtype=np.uint8)).astype(bool)


def masked_weight(W_bits: np.ndarray, B: np.ndarray, g_out: int = 1, g_in: int = G_IN) -> np.ndarray:
    """W_hat = W (.) M in float64 (Eq. 1); pruned entries are +0.0."""
    W = _bf16_to_f64(W_bits)
    M = expand_mask(B, g_out, g_in)
    if M.shape != W.shape:
        raise ValueError(f"mask expands to {M.shape}, weight is {W.shape}")
    return np.where(M, W, 0.0)


def masked_weight_bits(W_bits: np.ndarray, B: np.ndarray, g_out: int = 1, g_in: int = G_IN) -> np.ndarray:
    """W_hat as bf16 bits: W's bits where kept, 0x0000 (+0.0) where pruned."""
    W_bits = np.asarray(W_bits, dtype=np.uint16)
    M = expand_mask(B, g_out, g_in)
    return np.where(M, W_bits, np.uint16(0)).astype(np.uint16)


# ---------------------------------------------------------------------------
# the layer: y = x W_hat^T
# ---------------------------------------------------------------------------

def linear(x_bits: np.ndarray, W_bits: np.ndarray, B: np.ndarray, g_out: int = 1,
           g_in: int = G_IN) -> Tuple[np.ndarray, np.ndarray]:
    """y[t, r] = sum_k x[t, k] W_hat[r, k] in float64, and the magnitude sum
    A[t, r] = sum_k |x[t, k] W_hat[r, k]| that scales the acceptance bound.

    x_bits: uint16 [T, in] bf16 bits; W_bits: uint16 [out, in];
    B: [out/g_out, in/g_in] (default 1x256 groups: [out, in/256]).
    """
    x = _bf16_to_f64(x_bits)
    What = masked_weight(W_bits, B, g_out, g_in)
    if x.ndim != 2 or x.shape[1] != What.shape[1]:
        raise ValueError("x must be [T, in]")
    y = x @ What.T
    A = np.abs(x) @ np.abs(What).T
    return y, A


def linear_tokens(x_bits: np.ndarray, W_bits: np.ndarray, B: np.ndarray,
                  tokens: Sequence[int], g_out: int = 1, g_in: int = G_IN) -> Tuple[np.ndarray, np.ndarray]:
    """`linear` restricted to the listed token rows of x."""
    idx = np.asarray(list(tokens), dtype=np.int64)
    return linear(np.asarray(x_bits)[idx], W_bits, B, g_out, g_in)


# ---------------------------------------------------------------------------
# Eq. 2: sparsity accounting
# ---------------------------------------------------------------------------

def layer_sparsity(B: np.ndarray) -> float:
    """s^l = 1 - sum_uv B_uv / (G_out G_in)."""
    B = (np.asarray(B) != 0)
    return 1.0 - float(B.sum()) / float(B.size)


def global_sparsity(Bs: Iterable[np.ndarray], shapes: Iterable[Tuple[int, int]]) -> float:
    """s = sum_l s^l d_out d_in / sum_l d_out d_in (parameter-weighted mean)."""
    num = 0.0
    den = 0.0
    for B, (d_out, d_in) in zip(Bs, shapes):
        num += layer_sparsity(B) * d_out * d_in
        den += d_out * d_in
    return num / den


def preserved_rate(B: np.ndarray, g_out: int = 1, g_in: int = G_IN) -> float:
    """Active weights / total weights after applying the binary mask (App. F)."""
    M = expand_mask(B, g_out, g_in)
    return float(M.sum()) / float(M.size)


# ---------------------------------------------------------------------------
# packed layout (chunk-major kept-row lists)
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class Packed:
    out: int
    inp: int
    offsets: np.ndarray     # int64 [G+1]; chunk c owns packed rows [offsets[c], offsets[c+1])
    row_idx: np.ndarray     # int32 [K]; ascending kept rows of each chunk
    tiles: np.ndarray       # uint16 [K, 256]; tiles[j] = W[row_idx[j], 256c : 256c+256]
    win_off16: np.ndarray   # int32 [G, nw16+1]; first packed row of window w (rows 16w..) in chunk c
    kmask16: np.ndarray     # uint16 [G, nw16]; bit i = row 16w+i kept in chunk c

    @property
    def G(self) -> int:
        return self.inp // G_IN

    @property
    def kept(self) -> int:
        return int(self.offsets[-1])


def pack(W_bits: np.ndarray, B: np.ndarray) -> Packed:
    """Chunk-major packing: for chunk c = 0..G-1, for row r = 0..out-1 in ascending
    order, if B[r, c] keeps the group, append r to the row list and the 256
    weights W[r, 256c : 256c+256] (bit copy) to the tiles."""
    W_bits = np.asarray(W_bits, dtype=np.uint16)
    keep = np.asarray(B) != 0
    out, inp = W_bits.shape
    if inp % G_IN != 0:
        raise ValueError("in must be a multiple of 256")
    G = inp // G_IN
    if keep.shape != (out, G):
        raise ValueError("mask must be [out, in/256]")
    rows: List[int] = []
    tiles: List[np.ndarray] = []
    offsets = [0]
    for c in range(G):
        for r in range(out):
            if keep[r, c]:
                rows.append(r)
                tiles.append(W_bits[r, G_IN * c: G_IN * (c + 1)])
        offsets.append(len(rows))
    nw16 = (out + WIN16 - 1) // WIN16
    win_off16 = np.zeros((G, nw16 + 1), dtype=np.int32)
    kmask16 = np.zeros((G, nw16), dtype=np.uint16)
    for c in range(G):
        pos = offsets[c]
        for w in range(nw16):
            win_off16[c, w] = pos
            bits = 0
            for i in range(WIN16):
                r = WIN16 * w + i
                if r < out and keep[r, c]:
                    bits |= 1 << i
                    pos += 1
            kmask16[c, w] = bits
        win_off16[c, nw16] = pos
        assert pos == offsets[c + 1]
    return Packed(out=out, inp=inp,
                  offsets=np.asarray(offsets, dtype=np.int64),
                  row_idx=np.asarray(rows, dtype=np.int32),
                  tiles=(np.stack(tiles) if tiles else np.zeros((0, G_IN), np.uint16)).astype(np.uint16),
                  win_off16=win_off16, kmask16=kmask16)


def unpack(p: Packed) -> np.ndarray:
    """Scatter the packed tiles back to a dense [out, in] bf16 matrix; groups that are
    not in the row lists stay +0.0 (0x0000)."""
    W = np.zeros((p.out, p.inp), dtype=np.uint16)
    for c in range(p.G):
        for j in range(int(p.offsets[c]), int(p.offsets[c + 1])):
            r = int(p.row_idx[j])
            W[r, G_IN * c: G_IN * (c + 1)] = p.tiles[j]
    return W


def linear_packed(x_bits: np.ndarray, p: Packed) -> np.ndarray:
    """y from the packed layout: for every kept group (c, row_idx[j]), add the float64
    dot product of its 256 weights with x[:, 256c : 256c+256]; groups are visited in
    packed order, the 256 products of one group are summed left to right."""
    x = _bf16_to_f64(x_bits)
    T = x.shape[0]
    y = np.zeros((T, p.out), dtype=np.float64)
    tiles = _bf16_to_f64(p.tiles)
    for c in range(p.G):
        xc = x[:, G_IN * c: G_IN * (c + 1)]
        for j in range(int(p.offsets[c]), int(p.offsets[c + 1])):
            r = int(p.row_idx[j])
            for t in range(T):
                acc = 0.0
                for k in range(G_IN):
                    acc += xc[t, k] * tiles[j, k]
                y[t, r] += acc
    return y


# ---------------------------------------------------------------------------
# Sec. 2.2 and App. F: selector export and preserved rates
# ---------------------------------------------------------------------------

def select_groups(logits: np.ndarray) -> np.ndarray:
    """Evaluation-time selectors from float32 selector logits (Sec. 2.2; App. F).

    The group is kept when sigmoid(l) > 1/2.  sigmoid is strictly increasing
    with sigmoid(0) = 1/2, so that test is exactly l > 0 on the float32 value
    (a float64 sigmoid would round to 1/2 for |l| below about 1e-16 and lose
    the sign).  +0, -0 and NaN prune; +inf keeps.  Returns uint8 0/1 of the
    logits' shape ([G_out, G_in] row-major for one layer).
    """
    lg = np.asarray(logits, dtype=np.float32).astype(np.float64)
    B = np.zeros(lg.shape, dtype=np.uint8)
    B[lg > 0.0] = 1
    return B


def kept_groups(B: np.ndarray) -> int:
    """Number of retained groups, sum_uv B_uv (the numerator of Eq. 2)."""
    return int((np.asarray(B) != 0).sum())


def global_preserved_rate(Bs: Iterable[np.ndarray], shapes: Iterable[Tuple[int, int]]) -> float:
    """Share of all target parameters kept: 1 - s with s from Eq. 2."""
    return 1.0 - global_sparsity(Bs, shapes)


def qkv_preserved_rate(B_q: np.ndarray, B_k: np.ndarray, B_v: np.ndarray,
                       g_out: int = 1, g_in: int = G_IN) -> float:
    """App. F: the Q, K and V projections are reported as the plain mean of their
    three preserved rates."""
    return (preserved_rate(B_q, g_out, g_in) + preserved_rate(B_k, g_out, g_in)
            + preserved_rate(B_v, g_out, g_in)) / 3.0


# ---------------------------------------------------------------------------
# other group shapes: Sec. 2.1 with general g_out x g_in groups; the shapes the
# paper evaluates (Sec. 3.5 ablation, App. E)
# ---------------------------------------------------------------------------

GROUP_SHAPES = ((1, 128), (1, 256), (16, 16), (32, 32), (64, 64), (128, 128))


def group_grid(out: int, inp: int, g_out: int, g_in: int) -> Tuple[int, int]:
    """(G_out, G_in) = (d_out / g_out, d_in / g_in); the groups tile W exactly."""
    if g_out <= 0 or g_in <= 0 or out % g_out or inp % g_in:
        raise ValueError(f"a {out} x {inp} weight is not tiled by {g_out} x {g_in} groups")
    return out // g_out, inp // g_in


@dataclasses.dataclass
class PackedGroups:
    out: int
    inp: int
    g_out: int
    g_in: int
    offsets: np.ndarray     # int64 [G_in+1]; group column v owns packed groups [offsets[v], offsets[v+1])
    block_row: np.ndarray   # int32 [K]; ascending kept group rows u of each group column
    tiles: np.ndarray       # uint16 [K, g_out, g_in]; tiles[j] = W[g_out u : g_out (u+1), g_in v : g_in (v+1)]

    @property
    def kept(self) -> int:
        return int(self.offsets[-1])


def pack_groups(W_bits: np.ndarray, B: np.ndarray, g_out: int, g_in: int) -> PackedGroups:
    """Column-major packing for any group shape: for group column v = 0..G_in-1, for
    group row u = 0..G_out-1 in ascending order, if B[u, v] keeps the group, append u
    and the g_out x g_in block of W it covers (bit copy).  With g_out = 1 this is the
    chunk-major layout of `pack` (block_row = row_idx, tiles of one row)."""
    W_bits = np.asarray(W_bits, dtype=np.uint16)
    keep = np.asarray(B) != 0
    out, inp = W_bits.shape
    Go, Gi = group_grid(out, inp, g_out, g_in)
    if keep.shape != (Go, Gi):
        raise ValueError(f"mask must be [{Go}, {Gi}]")
    rows: List[int] = []
    tiles: List[np.ndarray] = []
    offsets = [0]
    for v in range(Gi):
        for u in range(Go):
            if keep[u, v]:
                rows.append(u)
                tiles.append(W_bits[g_out * u: g_out * (u + 1), g_in * v: g_in * (v + 1)])
        offsets.append(len(rows))
    return PackedGroups(out=out, inp=inp, g_out=g_out, g_in=g_in,
                        offsets=np.asarray(offsets, dtype=np.int64),
                        block_row=np.asarray(rows, dtype=np.int32),
                        tiles=(np.stack(tiles) if tiles else np.zeros((0, g_out, g_in), np.uint16)).astype(np.uint16))


def unpack_groups(p: PackedGroups) -> np.ndarray:
    """Scatter the packed blocks back to a dense [out, in] bf16 matrix; pruned groups
    stay +0.0 (0x0000)."""
    W = np.zeros((p.out, p.inp), dtype=np.uint16)
    Gi = p.inp // p.g_in
    for v in range(Gi):
        for j in range(int(p.offsets[v]), int(p.offsets[v + 1])):
            u = int(p.block_row[j])
            W[p.g_out * u: p.g_out * (u + 1), p.g_in * v: p.g_in * (v + 1)] = p.tiles[j]
    return W


def linear_packed_groups(x_bits: np.ndarray, p: PackedGroups) -> np.ndarray:
    """y from the packed blocks: for every kept group (u, v), y[:, rows of u] +=
    x[:, columns of v] . block^T in float64, groups visited in packed order."""
    x = _bf16_to_f64(x_bits)
    y = np.zeros((x.shape[0], p.out), dtype=np.float64)
    tiles = _bf16_to_f64(p.tiles.reshape(-1)).reshape(p.tiles.shape)
    Gi = p.inp // p.g_in
    for v in range(Gi):
        xv = x[:, p.g_in * v: p.g_in * (v + 1)]
        for j in range(int(p.offsets[v]), int(p.offsets[v + 1])):
            u = int(p.block_row[j])
            y[:, p.g_out * u: p.g_out * (u + 1)] += xv @ tiles[j].T
    return y


# ---------------------------------------------------------------------------
# Sec. 2.2: Gumbel-Sigmoid relaxation with a straight-through estimator (the
# training-side masked linear).  The paper names the relaxation (temperature
# T = 0.4 in Table 7) and the estimator without printing formulas; the
# standard form is used.  A sample draws two independent standard Gumbel
# variables per selector; their difference L is a standard logistic variable,
# passed in as `noise`.
#   forward:  B = [sigmoid((l + L) / tau) > 1/2] = [l + L > 0]  (binary, used
#             in W_hat = W (.) (B (x) 1) as in Eq. 1)
#   backward: dB/dl is replaced by d sigmoid((l + L) / tau) / dl
#             = s (1 - s) / tau with s = sigmoid((l + L) / tau); since
#             1 - sigmoid(a) = sigmoid(-a), it is evaluated as
#             sigmoid(a) sigmoid(-a) / tau, a = (l + L) / tau, which has no
#             cancellation where s is near 0 or 1
# ---------------------------------------------------------------------------

def gumbel_select(logits: np.ndarray, noise: np.ndarray, tau: float) -> Tuple[np.ndarray, np.ndarray]:
    """Binary selectors and their relaxation for one Gumbel-Sigmoid sample.

    l + L is formed in float32 (the sum both the oracle and the kernel decide
    on); B = [l + L > 0] (NaN prunes); s = sigmoid((l + L) / tau) in float64.
    Returns (B uint8, s float64), both of the logits' shape."""
    if not tau > 0:
        raise ValueError("tau must be positive")
    z32 = np.asarray(logits, dtype=np.float32) + np.asarray(noise, dtype=np.float32)
    B = (z32.astype(np.float64) > 0.0).astype(np.uint8)
    z = z32.astype(np.float64) / float(tau)
    with np.errstate(over="ignore"):
        s = 1.0 / (1.0 + np.exp(-z))
    return B, s


def gumbel_dsdl(logits: np.ndarray, noise: np.ndarray, tau: float) -> np.ndarray:
    """The straight-through derivative ds/dl = sigmoid(a) sigmoid(-a) / tau,
    a = (l + L) / tau, with l + L formed in float32 as in `gumbel_select`;
    float64 of the logits' shape."""
    if not tau > 0:
        raise ValueError("tau must be positive")
    z32 = np.asarray(logits, dtype=np.float32) + np.asarray(noise, dtype=np.float32)
    a = z32.astype(np.float64) / float(tau)
    with np.errstate(over="ignore"):
        return (1.0 / (1.0 + np.exp(-a))) * (1.0 / (1.0 + np.exp(a))) / float(tau)


def group_weight_grad(x_bits: np.ndarray, W_bits: np.ndarray, dy: np.ndarray, g_out: int = 1,
                      g_in: int = G_IN) -> np.ndarray:
    """dL/dB for every group (kept or pruned): with y = x W_hat^T, dL/dW_hat = dy^T x,
    and W_hat = W (.) (B (x) 1) gives dL/dB[u, v] = sum over the group's cells of
    W[r, k] (dy^T x)[r, k].  dy: float [T, out]."""
    x = _bf16_to_f64(x_bits)
    W = _bf16_to_f64(W_bits)
    dWhat = np.asarray(dy, dtype=np.float64).T @ x
    P = W * dWhat
    out, inp = W.shape
    Go, Gi = group_grid(out, inp, g_out, g_in)
    return P.reshape(Go, g_out, Gi, g_in).sum(axis=(1, 3))


def masked_linear_backward(x_bits: np.ndarray, W_bits: np.ndarray, B: np.ndarray, dy: np.ndarray,
                           dsdl: np.ndarray, g_out: int = 1,
                           g_in: int = G_IN) -> Tuple[np.ndarray, np.ndarray]:
    """Straight-through backward of y = x W_hat^T: the selector-logit gradient
    dL/dl = dL/dB * ds/dl (ds/dl from `gumbel_dsdl`) and the input gradient
    dL/dx = dy W_hat (W is frozen, so there is no weight gradient).
    Returns (dlogits, dx)."""
    G = group_weight_grad(x_bits, W_bits, dy, g_out, g_in)
    dlogits = G * np.asarray(dsdl, dtype=np.float64)
    dx = np.asarray(dy, dtype=np.float64) @ masked_weight(W_bits, B, g_out, g_in)
    return dlogits, dx
