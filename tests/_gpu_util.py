"""Helpers shared by the GPU parity tests (tensor marshalling and the acceptance bound)."""
import numpy as np

from oracle import groupsparse_oracle as orc

# Acceptance bound on y (per element): |y_gpu - y_oracle| <= 2^-7 * sum_kept |x w| + 1e-6.
# bf16 output rounding contributes at most 2^-9 |y| <= 2^-9 A, fp32 accumulation
# about K * 2^-24 A, so any fp32-accumulating order passes; bf16 accumulation fails.
REL = 2.0 ** -7
ABS = 1e-6


def to_dev(bits: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def to_bits(t) -> np.ndarray:
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def assert_within_bound(y_bits, x_bits, W_bits, B, tokens=None, what=""):
    if tokens is None:
        yr, A = orc.linear(x_bits, W_bits, B)
        yg = bf16_to_f64(y_bits)
    else:
        yr, A = orc.linear_tokens(x_bits, W_bits, B, tokens)
        yg = bf16_to_f64(y_bits[np.asarray(tokens)])
    err = np.abs(yg - yr)
    bound = REL * A + ABS
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {int(bad.sum())} elements outside the bound; first at {tuple(i)}: "
                             f"gpu {yg[tuple(i)]!r} oracle {yr[tuple(i)]!r} A {A[tuple(i)]!r}")
    return float((err / bound).max()) if err.size else 0.0


def sample_tokens(T: int, seed: int = 0, n_random: int = 12):
    base = {0, min(1, T - 1), T // 2, T - 1}
    rng = np.random.default_rng(seed)
    base.update(int(v) for v in rng.integers(0, T, size=n_random))
    return sorted(base)
