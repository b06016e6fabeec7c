"""Seeded synthetic inputs for the group-sparse linear layer.

This module only draws inputs: frozen bf16 weights W[out, in], per-group keep
masks B[out, in/256] and activations x[T, in].  It computes nothing of the
layer itself (no mask expansion, no products, no packing), so the CPU oracle
and the CUDA path can both be fed from it without sharing any of the method's
arithmetic.

Workload shapes follow the linear projections of a Transformer block (the
paper's target layers, Sec. 2.1 and Sec. 3.1): LLaMA-2-7B, LLaMA-2-13B and
Qwen2.5-7B projection shapes.  Values are synthetic: W ~ N(0, 0.02^2) rounded
to bf16, x ~ N(0, 1) rounded to bf16.  Groups are 1x256 along the input
dimension (the paper's default group shape, Sec. 2.1 and Table 7).  The
per-layer keep ratios vary under one global budget, which is the
layer-adaptive allocation the method learns (Sec. 2.3, Eq. 2); here the ratios
are drawn at random and rescaled so the global kept-group count is exact.

Seeding: every stream is a numpy PCG64 generator seeded with
SeedSequence([cfg_id, variant, layer_id, stream_id, *extra]); stream ids are
0 = W, 1 = per-layer ratios, 2 = group scores, 3 = x, 4 = outlier channels,
5 = selector logits.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Sequence, Tuple

import numpy as np

GROUP_IN = 256          # g_in of the 1x256 group shape (Sec. 2.1)

STREAM_W, STREAM_RATIOS, STREAM_SCORES, STREAM_X, STREAM_OUTLIERS, STREAM_LOGITS = 0, 1, 2, 3, 4, 5


# --------------------------------------------------------------------------
# bf16 bit helpers (conversions only)
# --------------------------------------------------------------------------

def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 with round-to-nearest-even; returns uint16 bits."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    rounding = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bits (uint16) to float32 exactly."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bits (uint16) to float64 exactly."""
    return bf16_bits_to_f32(b).astype(np.float64)


# --------------------------------------------------------------------------
# seeding
# --------------------------------------------------------------------------

def rng(cfg_id: int, variant: int, layer_id: int, stream_id: int, *extra: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([int(cfg_id), int(variant), int(layer_id), int(stream_id), *map(int, extra)])))


def seed_u64(cfg_id: int, variant: int, layer_id: int, stream_id: int, *extra: int) -> int:
    """A 63-bit integer seed derived from the same SeedSequence (for torch generators)."""
    ss = np.random.SeedSequence([int(cfg_id), int(variant), int(layer_id), int(stream_id), *map(int, extra)])
    return int(ss.generate_state(1, np.uint64)[0] & np.uint64((1 << 63) - 1))


# --------------------------------------------------------------------------
# workload shapes
# --------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Layer:
    name: str
    out: int
    inp: int

    @property
    def G(self) -> int:
        return self.inp // GROUP_IN

    @property
    def groups(self) -> int:
        return self.out * self.G


def _block(hidden: int, inter: int, kv: Optional[int] = None) -> List[Tuple[str, int, int]]:
    kv = hidden if kv is None else kv
    return [("q_proj", hidden, hidden), ("k_proj", kv, hidden), ("v_proj", kv, hidden),
            ("o_proj", hidden, hidden), ("gate_proj", inter, hidden), ("up_proj", inter, hidden),
            ("down_proj", hidden, inter)]


LLAMA2_7B_BLOCK = _block(4096, 11008)
LLAMA2_13B_BLOCK = _block(5120, 13824)
QWEN25_7B_BLOCK = _block(3584, 18944, kv=512)


@dataclasses.dataclass(frozen=True)
class Workload:
    """One seeded workload: a list of layers, their keep budgets and the token counts."""
    cfg_id: int
    name: str
    layers: Tuple[Layer, ...]
    density: float                      # global kept-group fraction
    ratio_range: Optional[Tuple[float, float]]   # per-layer keep ratio U[a, b] before rescaling
    tokens: Tuple[int, ...]
    outlier_frac: float = 0.0           # fraction of input channels scaled x20
    variant: int = 0
    allocation: str = "random"          # "random": U[a, b] ratios; "paper": paper_shaped_ratios

    @property
    def total_groups(self) -> int:
        return sum(l.groups for l in self.layers)

    @property
    def budget(self) -> int:
        return int(math.floor(self.density * self.total_groups + 0.5))


def _stack(block, nblocks: int) -> Tuple[Layer, ...]:
    return tuple(Layer(f"blk{b}.{n}", o, i) for b in range(nblocks) for (n, o, i) in block)


def workload(cfg_id: int, density: float = 0.5, blocks: Optional[int] = None,
             allocation: str = "random") -> Workload:
    """The five seeded workloads.

    1: one 1024x1024 layer, exactly half its 4096 groups kept, T = 8.
    2: one LLaMA-2-7B block (7 projections), per-module keep U[0.3, 0.7] rescaled to
       exactly 50 %, T in {1, 4, 16}.
    3: 32 LLaMA-2-7B blocks, per-layer U[0.2, 0.8] rescaled to 50 %, T = 2048 with 1 %
       of input channels scaled x20.
    4: 40 LLaMA-2-13B blocks, per-layer U[0.2, 0.8] rescaled to 50 %,
       T in {1, 16, 128, 512, 2048}.
    5: 28 Qwen2.5-7B blocks, global density d in {0.3, 0.5, 0.7} with per-layer
       U[d-0.2, d+0.2] rescaled to d, T in {1, 1024}.
    `blocks` truncates a stack to its first blocks (same seeds per layer index).
    allocation="paper" (workload 3 only) replaces the random ratios by
    paper_shaped_ratios, with their own seeds (variant 1).
    """
    if allocation not in ("random", "paper"):
        raise ValueError(f"unknown allocation {allocation!r}")
    if allocation == "paper":
        if cfg_id != 3:
            raise ValueError("the paper-shaped allocation is defined for the LLaMA-2-7B stack (workload 3)")
        n = 32 if blocks is None else blocks
        return Workload(3, f"llama2-7b-stack{n}-paper-alloc", _stack(LLAMA2_7B_BLOCK, n), 0.5, None, (1, 16, 2048),
                        outlier_frac=0.01, variant=1, allocation="paper")
    if cfg_id == 1:
        return Workload(1, "single-1024x1024", (Layer("linear", 1024, 1024),), 0.5, None, (8,))
    if cfg_id == 2:
        return Workload(2, "llama2-7b-block", _stack(LLAMA2_7B_BLOCK, 1), 0.5, (0.3, 0.7), (1, 4, 16))
    if cfg_id == 3:
        n = 32 if blocks is None else blocks
        return Workload(3, f"llama2-7b-stack{n}", _stack(LLAMA2_7B_BLOCK, n), 0.5, (0.2, 0.8), (2048,),
                        outlier_frac=0.01)
    if cfg_id == 4:
        n = 40 if blocks is None else blocks
        return Workload(4, f"llama2-13b-stack{n}", _stack(LLAMA2_13B_BLOCK, n), 0.5, (0.2, 0.8),
                        (1, 16, 128, 512, 2048))
    if cfg_id == 5:
        n = 28 if blocks is None else blocks
        d = float(density)
        return Workload(5, f"qwen2.5-7b-stack{n}-d{d:.1f}", _stack(QWEN25_7B_BLOCK, n), d,
                        (d - 0.2, d + 0.2), (1, 1024), variant=int(round(d * 100)))
    raise ValueError(f"unknown workload {cfg_id}")


# --------------------------------------------------------------------------
# keep budgets per layer
# --------------------------------------------------------------------------

def allocate_keep_counts(groups: Sequence[int], ratios: Sequence[float], budget: int) -> np.ndarray:
    """Integer kept-group counts k_l with sum(k_l) == budget and 0 <= k_l <= N_l.

    The drawn ratios r_l are rescaled by one factor alpha (bisection) so that
    sum(min(1, alpha*r_l) * N_l) reaches the budget from below; the floors are
    then topped up one group at a time in descending order of their fractional
    parts (ties: lower layer index), skipping layers that are already full.
    """
    N = np.asarray(groups, dtype=np.int64)
    r = np.asarray(ratios, dtype=np.float64)
    if budget < 0 or budget > int(N.sum()):
        raise ValueError("budget outside [0, total groups]")
    if np.any(r <= 0):
        raise ValueError("keep ratios must be positive")

    def kept(alpha: float) -> float:
        return float(np.sum(np.minimum(1.0, alpha * r) * N))

    lo, hi = 0.0, float(1.0 / r.min())
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if kept(mid) <= budget:
            lo = mid
        else:
            hi = mid
    exact = np.minimum(1.0, lo * r) * N
    k = np.floor(exact).astype(np.int64)
    k = np.minimum(k, N)
    rem = int(budget - k.sum())
    frac = exact - k
    order = sorted(range(len(N)), key=lambda i: (-frac[i], i))
    while rem > 0:
        progressed = False
        for i in order:
            if rem == 0:
                break
            if k[i] < N[i]:
                k[i] += 1
                rem -= 1
                progressed = True
        if not progressed:
            raise RuntimeError("cannot place the remaining budget")
    assert int(k.sum()) == budget and np.all(k >= 0) and np.all(k <= N)
    return k


def paper_shaped_ratios(nblocks: int = 32) -> np.ndarray:
    """Per-projection keep ratios [nblocks * 7] (q, k, v, o, gate, up, down per block)
    shaped after the learned LLaMA-2-7B allocation the paper describes in Sec. 3.5
    (only aggregate statistics are printed; the per-layer values are a figure):
    attention about 36.6 % and MLP about 56.6 % of their parameters, the down
    projection about 30.5 % of all preserved parameters, Q and K equal, V about 2.2x
    Q, O the largest attention projection, attention comparable to MLP in blocks
    3-17, and Q/K near 8 % with down above 53 % in blocks 22-31.  The depth profile
    is defined on 32 blocks; a shorter stack takes its first blocks.
    """
    q = np.empty(32)
    for b in range(32):
        if b < 3:
            q[b] = 0.20
        elif b <= 17:
            q[b] = 0.30
        elif b <= 21:
            q[b] = 0.25 - 0.05 * (b - 18)
        else:
            q[b] = 0.08
    v = 2.2 * q
    o = v + 0.14
    gate = np.full(32, 0.50)
    down = np.where(np.arange(32) >= 22, 0.81, 0.63)
    R = np.stack([q, q, v, o, gate, gate, down], axis=1)
    if not 1 <= nblocks <= 32:
        raise ValueError("the paper-shaped profile covers 1..32 blocks")
    return R[:nblocks].reshape(-1)


def keep_counts(wl: Workload) -> np.ndarray:
    """Per-layer kept-group counts of a workload (exact global budget)."""
    if wl.allocation == "paper":
        ratios = paper_shaped_ratios(len(wl.layers) // 7)
    elif wl.ratio_range is None:
        ratios = np.full(len(wl.layers), wl.density)
    else:
        a, b = wl.ratio_range
        ratios = rng(wl.cfg_id, wl.variant, 0, STREAM_RATIOS).uniform(a, b, size=len(wl.layers))
    return allocate_keep_counts([l.groups for l in wl.layers], ratios, wl.budget)


# --------------------------------------------------------------------------
# per-layer tensors (host, numpy)
# --------------------------------------------------------------------------

def group_mask(wl: Workload, layer_id: int, k: int) -> np.ndarray:
    """uint8 [out, G] keep mask with exactly k ones: the top-k of seeded U[0,1) scores
    (ties broken towards the lower flat index r*G + c)."""
    L = wl.layers[layer_id]
    scores = rng(wl.cfg_id, wl.variant, layer_id, STREAM_SCORES).random(L.groups)
    order = np.argsort(-scores, kind="stable")
    m = np.zeros(L.groups, dtype=np.uint8)
    m[order[:k]] = 1
    return m.reshape(L.out, L.G)


def group_mask_shaped(wl: Workload, layer_id: int, k: int, g_out: int, g_in: int) -> np.ndarray:
    """uint8 [out/g_out, in/g_in] keep mask for g_out x g_in groups that keeps the
    same fraction of the layer's groups as k of its 1x256 groups (rounded to the
    nearest whole group): the top of seeded U[0,1) scores, ties to the lower flat
    index.  The layer's shape must be tiled by the group."""
    L = wl.layers[layer_id]
    if L.out % g_out or L.inp % g_in:
        raise ValueError(f"{L.out}x{L.inp} is not tiled by {g_out}x{g_in} groups")
    Go, Gi = L.out // g_out, L.inp // g_in
    n = Go * Gi
    kk = int(math.floor(k * n / L.groups + 0.5))
    scores = rng(wl.cfg_id, wl.variant, layer_id, STREAM_SCORES, g_out, g_in).random(n)
    order = np.argsort(-scores, kind="stable")
    m = np.zeros(n, dtype=np.uint8)
    m[order[:kk]] = 1
    return m.reshape(Go, Gi)


def weight_bits(wl: Workload, layer_id: int) -> np.ndarray:
    """bf16 bits uint16 [out, in] of W ~ N(0, 0.02^2)."""
    L = wl.layers[layer_id]
    z = rng(wl.cfg_id, wl.variant, layer_id, STREAM_W).standard_normal((L.out, L.inp), dtype=np.float32)
    return f32_to_bf16_bits(z * np.float32(0.02))


def outlier_channels(wl: Workload, layer_id: int) -> np.ndarray:
    L = wl.layers[layer_id]
    n = int(math.floor(wl.outlier_frac * L.inp + 0.5))
    if n == 0:
        return np.zeros(0, dtype=np.int64)
    return np.sort(rng(wl.cfg_id, wl.variant, layer_id, STREAM_OUTLIERS).permutation(L.inp)[:n])


def activation_bits(wl: Workload, layer_id: int, T: int) -> np.ndarray:
    """bf16 bits uint16 [T, in] of x ~ N(0, 1); outlier channels (if any) scaled x20."""
    L = wl.layers[layer_id]
    z = rng(wl.cfg_id, wl.variant, layer_id, STREAM_X, T).standard_normal((T, L.inp), dtype=np.float32)
    xb = f32_to_bf16_bits(z)
    ch = outlier_channels(wl, layer_id)
    if ch.size:
        xb[:, ch] = f32_to_bf16_bits(bf16_bits_to_f32(xb[:, ch]) * np.float32(20.0))
    return xb


def random_mask(out: int, G: int, density: float, seed: int) -> np.ndarray:
    """uint8 [out, G] mask with each group kept independently with probability `density`."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([9001, seed])))
    return (g.random((out, G)) < density).astype(np.uint8)


def random_weight_bits(out: int, inp: int, seed: int, std: float = 0.02) -> np.ndarray:
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([9002, seed])))
    return f32_to_bf16_bits(g.standard_normal((out, inp), dtype=np.float32) * np.float32(std))


def random_activation_bits(T: int, inp: int, seed: int) -> np.ndarray:
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([9003, seed])))
    return f32_to_bf16_bits(g.standard_normal((T, inp), dtype=np.float32))


# --------------------------------------------------------------------------
# selector logits (the float32 scores a trained mask generator exports)
# --------------------------------------------------------------------------

# float32 bit patterns placed among synthetic logits: +-0, the smallest
# subnormals, the smallest normal, +-inf, quiet NaNs of both signs, +-max
SPECIAL_LOGIT_BITS = (0x00000000, 0x80000000, 0x00000001, 0x80000001, 0x00800000,
                      0x7F800000, 0xFF800000, 0x7FC00000, 0xFFC00000, 0x7F7FFFFF, 0xFF7FFFFF)


def logit_mean(density: float) -> float:
    """The mean mu of N(mu, 1) logits of which a fraction `density` is positive."""
    from statistics import NormalDist
    d = min(max(float(density), 1e-9), 1.0 - 1e-9)
    return NormalDist().inv_cdf(d)


def selector_logits(shape, density: float, seed: int, special_every: int = 0) -> np.ndarray:
    """float32 logits ~ N(logit_mean(density), 1) of the given shape.  With
    special_every = s > 0, about one entry in s (seeded positions) is replaced by
    one of SPECIAL_LOGIT_BITS, cycling through the list."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([9004, STREAM_LOGITS, seed])))
    lg = (g.standard_normal(shape, dtype=np.float32) + np.float32(logit_mean(density))).astype(np.float32)
    if special_every > 0 and lg.size:
        flat = lg.reshape(-1)
        n = max(1, flat.size // special_every)
        pos = g.choice(flat.size, size=min(n, flat.size), replace=False)
        vals = np.array(SPECIAL_LOGIT_BITS, dtype=np.uint32).view(np.float32)
        flat[pos] = vals[np.arange(pos.size) % vals.size]
    return lg


def selector_logits_device(n: int, density: float, seed: int, device="cuda"):
    """`selector_logits` drawn on the device (torch Philox), no special values."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed_u64(9004, 0, 0, STREAM_LOGITS, seed))
    return torch.randn((n,), generator=g, device=device, dtype=torch.float32) + logit_mean(density)


# --------------------------------------------------------------------------
# device-side generation for full-size stacks (torch RNG; same distributions)
# --------------------------------------------------------------------------

def weight_device(wl: Workload, layer_id: int, device="cuda"):
    """W ~ N(0, 0.02^2) as a bf16 torch tensor drawn on the device (torch's Philox stream
    seeded from the same SeedSequence).  Used where the numpy draw would be too slow."""
    import torch
    L = wl.layers[layer_id]
    g = torch.Generator(device=device)
    g.manual_seed(seed_u64(wl.cfg_id, wl.variant, layer_id, STREAM_W, 1))
    z = torch.randn((L.out, L.inp), generator=g, device=device, dtype=torch.float32)
    return (z * 0.02).to(torch.bfloat16)


def activation_device(wl: Workload, layer_id: int, T: int, device="cuda"):
    import torch
    L = wl.layers[layer_id]
    g = torch.Generator(device=device)
    g.manual_seed(seed_u64(wl.cfg_id, wl.variant, layer_id, STREAM_X, T, 1))
    x = torch.randn((T, L.inp), generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    ch = outlier_channels(wl, layer_id)
    if ch.size:
        idx = torch.as_tensor(ch, device=device)
        x[:, idx] = (x[:, idx].float() * 20.0).to(torch.bfloat16)
    return x
