"""Failure paths of the library, exercised without faulting the GPU, and the
use of one packed handle from several streams at once.

* A bounded wait that runs out: the test hook makes the first CTA (or CTA
  pair) of the next decode or prefill launch wait on a library word that
  nothing ever sets, before it issues any copy or MMA.  The wait runs out,
  the launch records GS_ERR_DEVICE_TIMEOUT, gs_device_status reports it, and
  the next normal call on the same handle must again match the oracle (the
  skipped units leave split counters half counted, which the library re-zeroes
  once the timeout has been read).
* A device allocation that fails: the test hook makes the nth allocation of
  gs_pack fail.  gs_pack must return GS_ERR_OOM and give back every byte.
* Several streams: gs_linear on one handle from two streams with no ordering
  between them gives, on each stream, exactly the single-stream result.
"""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl
from tests._gpu_util import assert_within_bound, to_bits, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


def make(gs, out, inp, d, seed):
    import torch
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    B = wl.random_mask(out, inp // 256, d, seed=seed + 7)
    return Wb, B, gs.pack(to_dev(Wb), torch.from_numpy(B).cuda())


@pytest.mark.parametrize("T", [3, 16])
def test_decode_wait_timeout_then_recovery(gs, T):
    import torch
    # 4096 x 11008: every 64-row block's 43 chunks are split over several
    # units, so the skipped CTA leaves split counters and the ticket half counted
    Wb, B, p = make(gs, 4096, 11008, 0.5, 31 + T)
    xb = wl.random_activation_bits(T, 11008, seed=40 + T)
    x = to_dev(xb)
    assert gs.device_status() == gs.GS_OK
    gs.debug_inject_wait(gs.ALGO_DECODE, 1_000_000)   # 1 ms on a word nothing sets
    gs.linear(x, p, algo=gs.ALGO_DECODE)
    torch.cuda.synchronize()
    assert gs.device_status() == gs.GS_ERR_DEVICE_TIMEOUT
    assert gs.device_status() == gs.GS_OK             # reading the status cleared it
    for _ in range(2):
        y = gs.linear(x, p, algo=gs.ALGO_DECODE)
        assert_within_bound(to_bits(y), xb, Wb, B, what=f"decode after timeout T={T}")
    assert gs.device_status() == gs.GS_OK


def test_batched_decode_wait_timeout_then_recovery(gs):
    shapes = [(4096, 11008, 0.5, 51), (11008, 4096, 0.6, 52), (512, 4096, 0.3, 53)]
    layers = [make(gs, *s) for s in shapes]
    T = 4
    xbs = [wl.random_activation_bits(T, s[1], seed=60 + i) for i, s in enumerate(shapes)]
    xs = [to_dev(b) for b in xbs]
    import torch
    ys = [torch.empty((T, s[0]), dtype=torch.bfloat16, device="cuda") for s in shapes]
    gs.debug_inject_wait(gs.ALGO_DECODE, 1_000_000)
    gs.linear_batched_into(xs, [l[2] for l in layers], ys)
    assert gs.device_status() == gs.GS_ERR_DEVICE_TIMEOUT
    gs.linear_batched_into(xs, [l[2] for l in layers], ys)
    for (Wb, B, _), xb, y in zip(layers, xbs, ys):
        assert_within_bound(to_bits(y), xb, Wb, B, what="batched decode after timeout")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("T", [64, 300])
def test_prefill_wait_timeout_then_recovery(gs, T):
    # T = 64: single-CTA tiles; T = 300: CTA pairs (both CTAs of pair 0 skip)
    Wb, B, p = make(gs, 4096, 4096, 0.5, 70 + T)
    xb = wl.random_activation_bits(T, 4096, seed=80 + T)
    x = to_dev(xb)
    gs.debug_inject_wait(gs.ALGO_PREFILL, 1_000_000)
    gs.linear(x, p, algo=gs.ALGO_PREFILL)
    assert gs.device_status() == gs.GS_ERR_DEVICE_TIMEOUT
    y = gs.linear(x, p, algo=gs.ALGO_PREFILL)
    assert_within_bound(to_bits(y), xb, Wb, B, what=f"prefill after timeout T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("g,T", [(0, 300), (0, 64), (16, 300), (32, 100)])
def test_prefill_dense_wait_timeout_then_recovery(gs, g, T):
    # the zero-filled-window kernel: CTA pair 0 skips its units (at T = 64 and
    # 100 the one token tile's first window), then a clean launch matches the oracle
    import torch
    if g == 0:
        Wb, B, p = make(gs, 4096, 4096, 0.5, 75)
        gg = None
    else:
        Wb = wl.random_weight_bits(1024, 2048, seed=76)
        B = wl.random_mask(1024 // g, 2048 // g, 0.5, seed=77)
        p = gs.pack_groups(to_dev(Wb), torch.from_numpy(B).cuda(), g, g)
        gg = g
    xb = wl.random_activation_bits(T, Wb.shape[1], seed=78 + g)
    x = to_dev(xb)
    # squares 16x16 at T = 300 and 32x32 at T = 100: the same kernel
    algo = gs.ALGO_PREFILL_DENSE if g == 0 else gs.ALGO_AUTO
    gs.debug_inject_wait(gs.ALGO_PREFILL_DENSE, 1_000_000)
    gs.linear(x, p, algo=algo)
    assert gs.device_status() == gs.GS_ERR_DEVICE_TIMEOUT
    y = to_bits(gs.linear(x, p, algo=algo))
    if gg is None:
        assert_within_bound(y, xb, Wb, B, what="zero-filled prefill after timeout")
    else:
        yr, A = orc.linear(xb, Wb, B, gg, gg)
        assert np.all(np.abs(wl.bf16_bits_to_f32(y).astype(np.float64) - yr) <= 2.0 ** -7 * A + 1e-6)
    assert gs.device_status() == gs.GS_OK


def test_failed_allocation_returns_oom_and_frees_everything(gs):
    import torch
    out, inp = 2048, 4096
    Wb = wl.random_weight_bits(out, inp, seed=90)
    B = wl.random_mask(out, inp // 256, 0.5, seed=91)
    W = to_dev(Wb)
    mask = torch.from_numpy(B).cuda()
    gs.pack(W, mask).free()            # warm-up: the library's per-device flag exists from here on
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    failures = 0
    for nth in range(1, 16):
        gs.debug_fail_alloc(nth)
        try:
            p = gs.pack(W, mask)
        except gs.GroupSparseError as e:
            assert e.status == gs.GS_ERR_OOM, e
            failures += 1
            torch.cuda.synchronize()
            assert torch.cuda.mem_get_info()[0] == free0, f"allocation {nth}: bytes not given back"
            continue
        finally:
            gs.debug_fail_alloc(0)
        # nth is past the last allocation of gs_pack: the pack succeeds and is correct
        got = p.export()
        ref = orc.pack(Wb, B)
        assert np.array_equal(got["offsets"], ref.offsets) and np.array_equal(got["tiles"], ref.tiles)
        p.free()
        break
    assert failures >= 6                # every buffer gs_pack allocates was made to fail once
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0


def test_one_handle_on_two_streams_at_once(gs):
    import torch
    Wb, B, p = make(gs, 4096, 11008, 0.5, 95)   # split blocks: the scratch is in use
    T = 8
    xbs = [wl.random_activation_bits(T, 11008, seed=96 + i) for i in range(2)]
    xs = [to_dev(b) for b in xbs]
    ref = [to_bits(gs.linear(x, p, algo=gs.ALGO_DECODE)) for x in xs]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    ys = [[torch.empty((T, 4096), dtype=torch.bfloat16, device="cuda") for _ in range(12)] for _ in range(2)]
    torch.cuda.synchronize()
    for i in range(12):
        for k in range(2):
            with torch.cuda.stream(streams[k]):
                gs.linear_into(xs[k], p, ys[k][i], algo=gs.ALGO_DECODE)
    torch.cuda.synchronize()
    for k in range(2):
        assert_within_bound(ref[k], xbs[k], Wb, B, what=f"stream {k}")
        for i in range(12):
            assert np.array_equal(to_bits(ys[k][i]), ref[k]), (k, i)
    assert gs.device_status() == gs.GS_OK
