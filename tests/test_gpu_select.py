"""Selector export on the GPU (gs_select_groups) vs the CPU oracle, through the C ABI.

The mask bytes and the kept count must match the oracle's threshold
(sigmoid(l) > 1/2, Sec. 2.2 and App. F) bit for bit, including the float32
special values and ragged lengths; exported masks then pack exactly as the
oracle packs them.
"""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl
from tests._gpu_util import to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


def run(gs, lg):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(lg, dtype=np.float32)).cuda()
    mask, kept = gs.select_groups(t)
    torch.cuda.synchronize()
    return mask.cpu().numpy(), int(kept.cpu()[0])


# lengths around the 512-selector warp step and the 4096-selector block step,
# plus a LLaMA-2-7B block's 790,528 groups and a length above one full grid pass
LENGTHS = [1, 15, 16, 17, 511, 512, 513, 4095, 4096, 4097, 100_003, 790_528, 5_000_011]


@pytest.mark.parametrize("n", LENGTHS)
def test_select_bit_exact(gs, n):
    lg = wl.selector_logits((n,), 0.4, seed=n, special_every=97)
    ref = orc.select_groups(lg)
    got, kept = run(gs, lg)
    assert got.dtype == np.uint8
    assert np.array_equal(got, ref)
    assert kept == orc.kept_groups(ref)


def test_select_special_values_everywhere(gs):
    # every special value at every position of a warp step and of the ragged tail
    vals = np.array(wl.SPECIAL_LOGIT_BITS, dtype=np.uint32).view(np.float32)
    lg = np.resize(vals, 512 * 3 + 37).astype(np.float32)
    got, kept = run(gs, lg)
    ref = orc.select_groups(lg)
    assert np.array_equal(got, ref) and kept == int(ref.sum())


@pytest.mark.parametrize("d", [0.0, 1.0])
def test_select_all_pruned_and_all_kept(gs, d):
    lg = np.full((3000,), -1.0 if d == 0.0 else 1.0, np.float32)
    got, kept = run(gs, lg)
    assert kept == int(d * 3000) and np.all(got == int(d))


def test_select_empty(gs):
    import torch
    kept = torch.full((1,), 77, dtype=torch.int64, device="cuda")
    mask, kept = gs.select_groups(torch.empty((0,), dtype=torch.float32, device="cuda"), kept=kept)
    assert mask.numel() == 0 and int(kept.cpu()[0]) == 0


def test_select_into_views_and_counts_overwritten(gs):
    import torch
    lg = wl.selector_logits((2048,), 0.5, seed=3)
    t = torch.from_numpy(lg).cuda()
    mask = torch.full((2048,), 9, dtype=torch.uint8, device="cuda")
    kept = torch.full((4,), 123, dtype=torch.int64, device="cuda")
    gs.select_groups(t, mask=mask, kept=kept)
    gs.select_groups(t, mask=mask, kept=kept)          # a second call overwrites, never accumulates
    torch.cuda.synchronize()
    ref = orc.select_groups(lg)
    assert np.array_equal(mask.cpu().numpy(), ref)
    assert kept.cpu().tolist() == [int(ref.sum()), 123, 123, 123]


@pytest.mark.parametrize("out,inp,d,seed", [(4096, 4096, 0.35, 1), (11008, 4096, 0.6, 2), (300, 768, 0.5, 3)])
def test_export_then_pack_matches_oracle(gs, out, inp, d, seed):
    import torch
    lg = wl.selector_logits((out, inp // 256), d, seed=seed, special_every=61)
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    p = gs.pack_from_logits(to_dev(Wb), torch.from_numpy(lg).cuda())
    ref = orc.pack(Wb, orc.select_groups(lg))
    got = p.export()
    assert p.kept == ref.kept
    for key in ("offsets", "row_idx", "tiles", "win_off16", "kmask16"):
        assert np.array_equal(got[key], getattr(ref, key)), key


def test_preserved_report_of_a_block_matches_oracle(gs):
    import torch
    layers = wl.workload(2).layers
    Bs, kept, shapes, names = [], [], [], []
    for i, L in enumerate(layers):
        lg = wl.selector_logits((L.out, L.inp // 256), 0.2 + 0.1 * i, seed=100 + i)
        _, k = gs.select_groups(torch.from_numpy(lg).cuda())
        kept.append(int(k.cpu()[0]))
        Bs.append(orc.select_groups(lg))
        shapes.append((L.out, L.inp))
        names.append(L.name)
    assert names[:3] == ["blk0.q_proj", "blk0.k_proj", "blk0.v_proj"]
    rep = gs.preserved_report(kept, shapes, names)
    for n, B in zip(names, Bs):
        assert rep["layers"][n] == orc.preserved_rate(B)
    assert rep["global"] == pytest.approx(orc.global_preserved_rate(Bs, shapes), abs=1e-15)
    assert rep["qkv"] == {"blk0": pytest.approx(orc.qkv_preserved_rate(*Bs[:3]), abs=1e-15)}
