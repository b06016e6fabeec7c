"""Seeded workload generator: budgets, determinism, shapes (no method arithmetic here)."""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl


def test_config_group_counts_and_budgets():
    assert wl.workload(1).total_groups == 4096 and wl.workload(1).budget == 2048
    assert wl.workload(2).total_groups == 790528 and wl.workload(2).budget == 395264
    assert wl.workload(3).total_groups == 25296896 and wl.workload(3).budget == 12648448
    assert wl.workload(4).total_groups == 49561600 and wl.workload(4).budget == 24780800
    w5 = wl.workload(5, 0.5)
    assert w5.total_groups == 25489408
    for d in (0.3, 0.5, 0.7):
        assert wl.workload(5, d).budget == int(np.floor(d * 25489408 + 0.5))
    assert {l.G for l in wl.workload(5).layers[:7]} == {14, 74}


@pytest.mark.parametrize("cfg,d", [(1, 0.5), (2, 0.5), (3, 0.5), (4, 0.5), (5, 0.3), (5, 0.5), (5, 0.7)])
def test_keep_counts_hit_budget_exactly(cfg, d):
    w = wl.workload(cfg, d)
    k = wl.keep_counts(w)
    N = np.array([l.groups for l in w.layers])
    assert int(k.sum()) == w.budget
    assert np.all(k >= 0) and np.all(k <= N)
    if w.ratio_range is not None:
        # layer-adaptive: per-layer densities spread out around the global one
        dens = k / N
        assert dens.std() > 0.05
    assert np.array_equal(k, wl.keep_counts(w))     # deterministic


def test_allocation_edge_cases():
    assert wl.allocate_keep_counts([10, 10], [1.0, 1.0], 20).tolist() == [10, 10]
    assert wl.allocate_keep_counts([10, 10], [0.5, 0.5], 0).tolist() == [0, 0]
    k = wl.allocate_keep_counts([100, 10], [0.9, 0.9], 105)       # second layer saturates
    assert k.tolist() == [95, 10]
    with pytest.raises(ValueError):
        wl.allocate_keep_counts([10], [0.5], 11)


def test_block_masks_meet_budget_and_eq2():
    """Masks of the one-block workload keep exactly the allocated groups; the
    parameter-weighted sparsity of Eq. 2 then equals 1 - K*/N because every
    1x256 group holds the same number of weights."""
    w = wl.workload(2)
    k = wl.keep_counts(w)
    masks = [wl.group_mask(w, i, int(k[i])) for i in range(len(w.layers))]
    for m, ki, L in zip(masks, k, w.layers):
        assert m.shape == (L.out, L.G) and int(m.sum()) == ki
    s = orc.global_sparsity(masks, [(L.out, L.inp) for L in w.layers])
    assert s == pytest.approx(1.0 - w.budget / w.total_groups, abs=1e-12)
    assert np.array_equal(masks[0], wl.group_mask(w, 0, int(k[0])))


def test_weights_and_activations_distribution():
    w = wl.workload(1)
    Wb = wl.weight_bits(w, 0)
    W = wl.bf16_bits_to_f64(Wb)
    assert W.shape == (1024, 1024)
    assert abs(W.std() - 0.02) < 5e-4 and abs(W.mean()) < 1e-3
    xb = wl.activation_bits(w, 0, 8)
    assert xb.shape == (8, 1024)
    assert np.array_equal(Wb, wl.weight_bits(w, 0))


def test_outlier_channels():
    w = wl.workload(3, blocks=1)
    L = w.layers[0]
    ch = wl.outlier_channels(w, 0)
    assert ch.size == 41                    # 1 % of 4096 channels
    x = wl.bf16_bits_to_f64(wl.activation_bits(w, 0, 64))
    big = np.abs(x[:, ch]).mean()
    rest = np.abs(np.delete(x, ch, axis=1)).mean()
    assert 15 < big / rest < 25
    assert wl.outlier_channels(w, 6).size == 110   # down_proj: 1 % of 11008


def test_selector_logits_density_and_specials():
    lg = wl.selector_logits((400, 50), 0.3, seed=1)
    assert lg.dtype == np.float32 and lg.shape == (400, 50)
    assert abs(float((lg > 0).mean()) - 0.3) < 0.01
    assert np.array_equal(lg, wl.selector_logits((400, 50), 0.3, seed=1))       # seeded
    sp = wl.selector_logits((400, 50), 0.7, seed=2, special_every=50)
    bits = sp.view(np.uint32).reshape(-1)
    present = set(int(b) for b in bits) & set(wl.SPECIAL_LOGIT_BITS)
    assert present == set(wl.SPECIAL_LOGIT_BITS)
    assert np.isnan(sp).sum() >= 2


def test_paper_shaped_allocation_matches_printed_statistics():
    # Sec. 3.5 (LLaMA-2-7B, 50 % sparsity): attention 36.6 %, MLP 56.6 %, down 30.5 % of all
    # preserved parameters, Q/K about 8 % of groups and down above 53 % in blocks 22-31
    w = wl.workload(3, allocation="paper")
    k = wl.keep_counts(w).reshape(32, 7)
    N = np.array([L.groups for L in w.layers[:7]])
    assert int(k.sum()) == w.budget == w.total_groups // 2
    rate = k / N
    attn = k[:, :4].sum() / (N[:4].sum() * 32)
    mlp = k[:, 4:].sum() / (N[4:].sum() * 32)
    assert abs(attn - 0.366) < 0.005 and abs(mlp - 0.566) < 0.005
    assert abs(k[:, 6].sum() / k.sum() - 0.305) < 0.005
    assert np.all(np.abs(rate[22:, 0] - 0.08) < 0.01) and np.all(rate[22:, 6] > 0.53)
    assert np.all(np.abs(rate[:, 0] - rate[:, 1]) < 0.05) and np.all(np.abs(rate[:, 4] - rate[:, 5]) < 0.05)
    assert abs(rate[:, 2].sum() / rate[:, 0].sum() - 2.2) < 0.1
    assert np.all(rate[:, 3] >= rate[:, :3].max(axis=1))
    mid = slice(3, 18)
    assert abs(k[mid, :4].sum() / (N[:4].sum() * 15) - k[mid, 4:].sum() / (N[4:].sum() * 15)) < 0.1
    # masks of the variant differ from the random-allocation stack's, and are reproducible
    m = wl.group_mask(w, 0, int(k[0, 0]))
    assert int(m.sum()) == int(k[0, 0]) and np.array_equal(m, wl.group_mask(w, 0, int(k[0, 0])))
    with pytest.raises(ValueError):
        wl.workload(4, allocation="paper")


def test_every_config_shape_is_tiled_by_every_group_shape():
    for cfg, d in ((1, 0.5), (2, 0.5), (3, 0.5), (4, 0.5), (5, 0.5)):
        for L in wl.workload(cfg, d).layers[:7]:
            for g_out, g_in in orc.GROUP_SHAPES:
                Go, Gi = orc.group_grid(L.out, L.inp, g_out, g_in)
                assert Go * g_out == L.out and Gi * g_in == L.inp
