"""Training-side selectors (Sec. 2.2): the Gumbel-Sigmoid sample and the
straight-through backward of the masked linear, through the C ABI, against
the oracle.

The sample's mask and kept count must match exactly (both decide on the
float32 sum l + L); the estimator's derivative ds/dl = s (1 - s) / tau within
float32 rounding.  The logit
gradient must satisfy |dl - dl_oracle| <= 2^-10 * A + 1e-9 with A the same
sum over magnitudes (fp32 accumulation of bf16 products); the input gradient,
a bf16 output, the forward's bound 2^-7 * A + 1e-6.
"""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl
from tests._gpu_util import bf16_to_f64, to_bits, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


def logistic_noise(shape, seed):
    g = np.random.default_rng(seed)
    u = g.random(shape)
    return (np.log(u) - np.log1p(-u)).astype(np.float32)


@pytest.mark.parametrize("n,tau", [(1, 0.4), (1000, 0.4), (4096 * 43, 0.4), (77777, 2.0)])
def test_gumbel_select_matches_oracle(gs, n, tau):
    import torch
    lg = wl.selector_logits((n,), 0.5, seed=n, special_every=97 if n > 100 else 0)
    noise = logistic_noise(n, n + 1)
    mask, dsdl, kept = gs.gumbel_select(torch.from_numpy(lg).cuda(), torch.from_numpy(noise).cuda(), tau)
    B, s = orc.gumbel_select(lg, noise, tau)
    assert np.array_equal(mask.cpu().numpy(), B)
    assert int(kept.cpu()[0]) == int(B.sum())
    ref = orc.gumbel_dsdl(lg, noise, tau)
    dg = dsdl.cpu().numpy().astype(np.float64)
    fin = np.isfinite(ref) & (ref > 1e-30)            # away from float32 underflow
    assert np.allclose(dg[fin], ref[fin], rtol=2e-5, atol=0)


def backward_case(gs, out, inp, g_out, g_in, T, seed, want_dx=True):
    import torch
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    xb = wl.random_activation_bits(T, inp, seed=seed + 1)
    dyb = wl.random_activation_bits(T, out, seed=seed + 2)
    shape = (out // g_out, inp // g_in)
    lg = np.random.default_rng(seed + 3).standard_normal(shape).astype(np.float32)
    noise = logistic_noise(shape, seed + 4)
    tau = 0.4
    mask, dsdl, _ = gs.gumbel_select(torch.from_numpy(lg).cuda(), torch.from_numpy(noise).cuda(), tau)
    W = to_dev(Wb)
    p = gs.pack_groups(W, mask, g_out, g_in)
    dl, dx = gs.masked_linear_backward(to_dev(xb), W, p, to_dev(dyb), dsdl, want_dx=want_dx)
    B, _ = orc.gumbel_select(lg, noise, tau)
    assert np.array_equal(mask.cpu().numpy(), B)
    dy = bf16_to_f64(dyb)
    dsdl_ref = orc.gumbel_dsdl(lg, noise, tau)
    dl_ref, dx_ref = orc.masked_linear_backward(xb, Wb, B, dy, dsdl_ref, g_out, g_in)
    # magnitude sums for the bounds
    x, W64 = bf16_to_f64(xb), bf16_to_f64(Wb)
    Ag = (np.abs(W64) * (np.abs(dy).T @ np.abs(x))).reshape(shape[0], g_out, shape[1], g_in).sum(axis=(1, 3))
    A_dl = Ag * dsdl_ref
    err = np.abs(dl.cpu().numpy().astype(np.float64) - dl_ref)
    assert np.all(err <= 2.0 ** -10 * A_dl + 1e-9), f"dlogits: max excess {(err - 2.0 ** -10 * A_dl).max()}"
    if want_dx:
        A_dx = np.abs(dy) @ np.abs(orc.masked_weight(Wb, B, g_out, g_in))
        e2 = np.abs(bf16_to_f64(to_bits(dx)) - dx_ref)
        assert np.all(e2 <= 2.0 ** -7 * A_dx + 1e-6)
    return p


@pytest.mark.parametrize("g_out,g_in", [(1, 256), (1, 128), (16, 16), (32, 32), (128, 128)])
@pytest.mark.parametrize("T", [5, 64, 300])
def test_straight_through_backward(gs, g_out, g_in, T):
    backward_case(gs, 256, 512, g_out, g_in, T, seed=10 * T + g_in)


def test_backward_at_a_block_shape_without_dx(gs):
    backward_case(gs, 4096, 11008, 1, 256, 128, seed=77, want_dx=False)
    assert gs.device_status() == gs.GS_OK


def test_training_step_forward_uses_the_sampled_mask(gs):
    # forward of the step: pack W with the sample's mask, then gs_linear
    import torch
    out, inp, T = 1024, 2048, 40
    Wb = wl.random_weight_bits(out, inp, seed=5)
    xb = wl.random_activation_bits(T, inp, seed=6)
    lg = np.random.default_rng(7).standard_normal((out, inp // 256)).astype(np.float32)
    noise = logistic_noise(lg.shape, 8)
    mask, _, kept = gs.gumbel_select(torch.from_numpy(lg).cuda(), torch.from_numpy(noise).cuda(), 0.4)
    p = gs.pack(to_dev(Wb), mask)
    assert p.kept == int(kept.cpu()[0])
    y = to_bits(gs.linear(to_dev(xb), p))
    B, _ = orc.gumbel_select(lg, noise, 0.4)
    yr, A = orc.linear(xb, Wb, B)
    assert np.all(np.abs(bf16_to_f64(y) - yr) <= 2.0 ** -7 * A + 1e-6)
