"""gs_pack_index_noalloc: the packing index step without any device allocation.

Some callers cannot allocate device memory at the moment they pack weights:
code that runs while a CUDA graph is being captured (where cudaMalloc is not
allowed), or an inference runtime that hands every byte of device memory out
of its own fixed arena and forbids hidden allocations.  For them the library
exposes gs_pack_index_noalloc, which writes the same chunk offsets, window
offsets and window kept-masks as gs_pack into buffers the caller provides; its
temporary per-window counts live in a fixed array inside the library.

Each case calls the entry point twice in a row (the shared array keeps the
previous call's contents) and compares both results bit for bit with the CPU
oracle's packed layout for the same mask, and with what gs_pack produces.  One
case packs a large layer and then a smaller one with a different mask, so a
result that read counts left behind by the earlier call would differ.
"""
import ctypes

import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl

pytestmark = pytest.mark.gpu

GS_OK, GS_ERR_INVALID_ARG, GS_ERR_UNSUPPORTED = 0, 1, 2


@pytest.fixture(scope="module")
def ctx(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse as gs
    lib = ctypes.CDLL(str(built_lib))
    vp, i64 = ctypes.c_void_p, ctypes.c_int64
    lib.gs_pack_index_noalloc.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    lib.gs_pack_index_noalloc.restype = ctypes.c_int
    return torch, gs, lib


def run_noalloc(torch, lib, mask, out, inp):
    G = inp // 256
    nw16 = (out + 15) // 16
    offsets = torch.full((G + 1,), -1, dtype=torch.int64, device="cuda")
    win = torch.full((G * (nw16 + 1),), -1, dtype=torch.int32, device="cuda")
    km = torch.full((G * nw16,), -1, dtype=torch.int16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    st = lib.gs_pack_index_noalloc(mask.data_ptr(), out, inp, offsets.data_ptr(), win.data_ptr(), km.data_ptr(),
                                   stream)
    assert st == GS_OK, st
    torch.cuda.synchronize()
    return (offsets.cpu().numpy(), win.cpu().numpy().reshape(G, nw16 + 1),
            km.cpu().numpy().view(np.uint16).reshape(G, nw16))


@pytest.mark.parametrize("out,inp,d,seed", [(300, 768, 0.5, 1), (1024, 1024, 0.5, 2), (11008, 4096, 0.45, 3),
                                             (4096, 11008, 0.5, 4), (17, 256, 0.0, 5), (512, 3584, 1.0, 6)])
def test_matches_gs_pack_on_two_calls(ctx, out, inp, d, seed):
    torch, gs, lib = ctx
    B = wl.random_mask(out, inp // 256, d, seed=seed)
    Wb = wl.random_weight_bits(out, inp, seed=seed)
    mask = torch.from_numpy(B).cuda()
    W = torch.from_numpy(Wb.view(np.int16)).view(torch.bfloat16).cuda()
    ref = orc.pack(Wb, B)
    lib_ref = gs.pack(W, mask).export()
    for _ in range(2):
        offsets, win, km = run_noalloc(torch, lib, mask, out, inp)
        assert np.array_equal(offsets, ref.offsets)
        assert np.array_equal(win, ref.win_off16)
        assert np.array_equal(km, ref.kmask16)
        assert np.array_equal(offsets, lib_ref["offsets"])
        assert np.array_equal(win, lib_ref["win_off16"])
        assert np.array_equal(km, lib_ref["kmask16"])


def test_large_then_small_layer_with_another_mask(ctx):
    # the shared array still holds the large layer's counts when the small one
    # is packed; every entry the small call reads must be its own
    torch, gs, lib = ctx
    shapes = [(13824, 5120, 0.7, 11), (300, 1024, 0.3, 12), (13824, 5120, 0.2, 13), (48, 512, 0.9, 14)]
    for out, inp, d, seed in shapes:
        B = wl.random_mask(out, inp // 256, d, seed=seed)
        Wb = np.zeros((out, inp), np.uint16)
        ref = orc.pack(Wb, B)
        offsets, win, km = run_noalloc(torch, lib, torch.from_numpy(B).cuda(), out, inp)
        assert np.array_equal(offsets, ref.offsets), (out, inp)
        assert np.array_equal(win, ref.win_off16), (out, inp)
        assert np.array_equal(km, ref.kmask16), (out, inp)


def test_rejects_sizes_beyond_the_fixed_array(ctx):
    torch, gs, lib = ctx
    fake = 0x1000   # never dereferenced: the size check fails before any launch
    G = 64
    out = 16 * ((1 << 20) // G + 1)          # G * ceil(out/16) just above 2^20
    assert lib.gs_pack_index_noalloc(fake, out, 256 * G, fake, fake, fake, None) == GS_ERR_UNSUPPORTED
    assert lib.gs_pack_index_noalloc(None, 16, 256, fake, fake, fake, None) == GS_ERR_INVALID_ARG
    assert lib.gs_pack_index_noalloc(fake, 16, 300, fake, fake, fake, None) == GS_ERR_INVALID_ARG
    # misaligned outputs and overlapping buffers are refused before any launch
    m, o, w, k = 0x100000, 0x200000, 0x300000, 0x400000
    assert lib.gs_pack_index_noalloc(m, 16, 512, o + 4, w, k, None) == GS_ERR_INVALID_ARG
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w + 2, k, None) == GS_ERR_INVALID_ARG
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w, k + 1, None) == GS_ERR_INVALID_ARG
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, o + 16, k, None) == GS_ERR_INVALID_ARG
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w, m + 16, None) == GS_ERR_INVALID_ARG
