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
