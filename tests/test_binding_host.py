"""The Python binding rejects bad arguments before any device call (no GPU
needed): host tensors, wrong dtypes, shape mismatches, freed handles."""
import pytest
import torch


@pytest.fixture(scope="module")
def gs(built_lib):
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


def test_pack_rejects_host_tensors(gs):
    W = torch.zeros((4, 256), dtype=torch.bfloat16)
    M = torch.ones((4, 1), dtype=torch.uint8)
    with pytest.raises(ValueError, match="CUDA"):
        gs.pack(W, M)


def test_linear_rejects_host_and_mistyped_tensors(gs):
    p = gs.Packed(0, 4, 256)   # a null handle: never reached, the tensors fail first
    with pytest.raises(ValueError, match="CUDA"):
        gs.linear_into(torch.zeros((2, 256), dtype=torch.bfloat16), p,
                       torch.zeros((2, 4), dtype=torch.bfloat16))
    with pytest.raises(ValueError, match="CUDA"):
        gs.linear_into(torch.zeros((2, 256), dtype=torch.float32), p,
                       torch.zeros((2, 4), dtype=torch.bfloat16))


def test_batched_rejects_mismatched_lists(gs):
    p = gs.Packed(0, 4, 256)
    x = torch.zeros((2, 256), dtype=torch.bfloat16)
    y = torch.zeros((2, 4), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="same length"):
        gs.linear_batched_into([x, x], [p], [y, y])
    with pytest.raises(ValueError, match="CUDA"):
        gs.linear_batched_into([x], [p], [y])
    gs.linear_batched_into([], [], [])          # an empty batch is a no-op


def test_freed_handle_is_refused(gs):
    p = gs.Packed(0, 4, 256)
    with pytest.raises(ValueError, match="freed"):
        _ = p.handle
    p.free()                                    # freeing twice is harmless


def test_select_rejects_host_and_mistyped_tensors(gs):
    with pytest.raises(ValueError, match="CUDA"):
        gs.select_groups(torch.zeros((4, 2), dtype=torch.float32))
    with pytest.raises(ValueError, match="CUDA"):
        gs.select_groups(torch.zeros((4, 2), dtype=torch.float16))


def test_preserved_report_against_oracle():
    import numpy as np
    from oracle import groupsparse_oracle as orc
    from paper_2609_33977_gb300 import groupsparse as gs
    rng = np.random.default_rng(4)
    shapes = [(32, 512), (32, 512), (16, 512), (48, 1024), (8, 768)]
    names = ["b1.q_proj", "b1.k_proj", "b1.v_proj", "b1.o_proj", "b1.down_proj"]
    Bs = [(rng.random((o, i // 256)) < 0.4).astype(np.uint8) for o, i in shapes]
    rep = gs.preserved_report([int(B.sum()) for B in Bs], shapes, names)
    for n, B in zip(names, Bs):
        assert rep["layers"][n] == orc.preserved_rate(B)
    assert rep["global"] == pytest.approx(orc.global_preserved_rate(Bs, shapes), abs=1e-15)
    assert rep["qkv"] == {"b1": pytest.approx(orc.qkv_preserved_rate(*Bs[:3]), abs=1e-15)}
    # no complete q/k/v trio, no QKV entry; a count that cannot fit is refused
    assert gs.preserved_report([1], [(1, 256)], ["x.q"])["qkv"] == {}
    with pytest.raises(gs.GroupSparseError) as e:
        gs.preserved_report([3], [(2, 256)])
    assert e.value.status == gs.GS_ERR_INVALID_ARG
