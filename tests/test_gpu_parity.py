"""CUDA path vs the CPU oracle, through the C ABI (pack / linear / unpack).

Packing and unpacking must match bit for bit; y must satisfy
|y - y_oracle| <= 2^-7 * sum_kept |x w| + 1e-6 element-wise.
"""
import numpy as np
import pytest

from oracle import groupsparse_oracle as orc
from paper_2609_33977_gb300 import workload as wl
from tests._gpu_util import assert_within_bound, sample_tokens, to_bits, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gs(built_lib):
    import torch
    assert torch.cuda.is_available(), "the -m gpu tests need a CUDA device"
    from paper_2609_33977_gb300 import groupsparse
    return groupsparse


_cache = {}


def layer(out, inp, d, seed):
    key = (out, inp, d, seed)
    if key not in _cache:
        Wb = wl.random_weight_bits(out, inp, seed=seed)
        B = wl.random_mask(out, inp // 256, d, seed=seed + 1000)
        _cache[key] = (Wb, B)
    return _cache[key]


def packed(gs, Wb, B):
    import torch
    return gs.pack(to_dev(Wb), torch.from_numpy(np.ascontiguousarray(B, dtype=np.uint8)).cuda())


PACK_SHAPES = [(1, 256, 1.0, 1), (17, 512, 0.5, 2), (300, 768, 0.5, 3), (1024, 1024, 0.5, 4),
               (512, 3584, 0.3, 5), (4096, 4096, 0.5, 6), (11008, 4096, 0.45, 7), (4096, 11008, 0.5, 8),
               (129, 256, 0.0, 9), (200, 2048, 1.0, 10)]


@pytest.mark.parametrize("out,inp,d,seed", PACK_SHAPES)
def test_pack_and_unpack_bit_exact(gs, out, inp, d, seed):
    Wb, B = layer(out, inp, d, seed)
    p = packed(gs, Wb, B)
    ref = orc.pack(Wb, B)
    got = p.export()
    assert p.kept == ref.kept == int(B.sum())
    assert np.array_equal(got["offsets"], ref.offsets)
    assert np.array_equal(got["row_idx"], ref.row_idx)
    assert np.array_equal(got["tiles"], ref.tiles)
    assert np.array_equal(got["win_off16"], ref.win_off16)
    assert np.array_equal(got["kmask16"], ref.kmask16)
    assert np.array_equal(to_bits(gs.unpack(p)), orc.masked_weight_bits(Wb, B))


def test_pack_is_deterministic(gs):
    Wb, B = layer(4096, 4096, 0.5, 6)
    a = packed(gs, Wb, B).export()
    b = packed(gs, Wb, B).export()
    for k in a:
        assert np.array_equal(a[k], b[k]), k


DECODE_SHAPES = [(300, 768, 0.5, 3), (1024, 1024, 0.5, 4), (512, 3584, 0.3, 5), (4096, 4096, 0.5, 6),
                 (4096, 11008, 0.5, 8), (17, 512, 0.5, 2), (129, 256, 0.0, 9), (200, 2048, 1.0, 10)]
DECODE_T = list(range(1, 18)) + [24, 31, 32, 33, 64, 65, 100]


@pytest.mark.parametrize("out,inp,d,seed", DECODE_SHAPES)
def test_decode_parity(gs, out, inp, d, seed):
    Wb, B = layer(out, inp, d, seed)
    p = packed(gs, Wb, B)
    for T in DECODE_T:
        xb = wl.random_activation_bits(T, inp, seed=seed * 100 + T)
        y = gs.linear(to_dev(xb), p, algo=gs.ALGO_DECODE)
        assert_within_bound(to_bits(y), xb, Wb, B, what=f"decode {out}x{inp} d={d} T={T}")
    assert gs.device_status() == gs.GS_OK


PREFILL_SHAPES = [(300, 768, 0.5, 3), (1024, 1024, 0.5, 4), (640, 2560, 0.9, 11), (520, 512, 0.05, 12),
                  (256, 4096, 1.0, 13), (1000, 1280, 0.0, 14), (4096, 4096, 0.5, 6), (17, 512, 0.5, 2)]
PREFILL_T = [1, 7, 64, 127, 128, 129, 255, 256, 300, 513]


@pytest.mark.parametrize("out,inp,d,seed", PREFILL_SHAPES)
def test_prefill_parity(gs, out, inp, d, seed):
    Wb, B = layer(out, inp, d, seed)
    p = packed(gs, Wb, B)
    for T in PREFILL_T:
        xb = wl.random_activation_bits(T, inp, seed=seed * 100 + T + 7)
        y = gs.linear(to_dev(xb), p, algo=gs.ALGO_PREFILL)
        assert_within_bound(to_bits(y), xb, Wb, B, what=f"prefill {out}x{inp} d={d} T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("out,inp,d,seed", PREFILL_SHAPES)
def test_prefill_dense_parity(gs, out, inp, d, seed):
    """The zero-filled-window kernel: pruned rows multiply as zeros, so y keeps the same bound."""
    Wb, B = layer(out, inp, d, seed)
    p = packed(gs, Wb, B)
    for T in PREFILL_T:
        xb = wl.random_activation_bits(T, inp, seed=seed * 100 + T + 9)
        y = gs.linear(to_dev(xb), p, algo=gs.ALGO_PREFILL_DENSE)
        assert_within_bound(to_bits(y), xb, Wb, B, what=f"prefill-dense {out}x{inp} d={d} T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("go,gi", [(1, 256), (1, 128), (32, 32)])
def test_prefill_dense_large_ragged_layers(gs, go, gi):
    """Zero-filled kernel on ~10K-row layers at T ~ 1K (80+ units, more than one per CTA pair):
    every element against the oracle, ragged rows and tokens, an empty window between non-empty
    ones, and a batched call beside a small layer equal to single calls bit for bit."""
    import torch
    from tests._gpu_util import REL, ABS, bf16_to_f64
    inp = 512
    cases = []
    for out, d, seed in ((10240, 0.5, 61), (10304, 0.3, 62)):   # 10304: a 64-row last window
        Wb = wl.random_weight_bits(out, inp, seed=seed)
        B = wl.random_mask(out // go, inp // gi, d, seed=seed + 1000)
        if go == 1:
            B[512:768, :] = 0    # window 2 empty, windows 1 and 3 not
        else:
            B[512 // go:768 // go, :] = 0
        p = gs.pack_groups(to_dev(Wb), torch.from_numpy(np.ascontiguousarray(B, dtype=np.uint8)).cuda(), go, gi)
        cases.append((Wb, B, p))
    for T in (1000, 1024):
        for Wb, B, p in cases:
            xb = wl.random_activation_bits(T, inp, seed=T + Wb.shape[0])
            y = to_bits(gs.linear(to_dev(xb), p, algo=gs.ALGO_PREFILL_DENSE if go == 1 else gs.ALGO_AUTO))
            yr, A = orc.linear(xb, Wb, B, go, gi)
            err = np.abs(bf16_to_f64(y) - yr)
            assert np.all(err <= REL * A + ABS), (go, gi, Wb.shape, T, float((err / (REL * A + ABS)).max()))
    # batched: the large layer beside a small layer of the same group shape
    Ws = wl.random_weight_bits(512, inp, seed=63)
    Bs = wl.random_mask(512 // go, inp // gi, 0.5, seed=64)
    ps = gs.pack_groups(to_dev(Ws), torch.from_numpy(Bs).cuda(), go, gi)
    T = 1024
    layers = [(cases[0][0], cases[0][2]), (Ws, ps)]
    xbs = [wl.random_activation_bits(T, inp, seed=70 + i) for i in range(2)]
    ys = [torch.empty((T, W.shape[0]), dtype=torch.bfloat16, device="cuda") for W, _ in layers]
    gs.linear_batched_into([to_dev(b) for b in xbs], [p for _, p in layers], ys)   # AUTO: zero-filled kernel at T = 1024
    for (W, p), xb, y in zip(layers, xbs, ys):
        assert np.array_equal(to_bits(y), to_bits(gs.linear(to_dev(xb), p)))
    assert gs.device_status() == gs.GS_OK


def test_prefill_more_tiles_than_the_tile_list(gs):
    """Launches with more tiles than the balanced tile list holds (2048) fall back to the fixed
    stride: a 41120-row layer on the gathering kernel (8 x 257 tiles) and a 65792-row layer on the
    zero-filled kernel (8 x 257 units) at T = 2048, sampled tokens against the oracle."""
    T = 2048
    for out, algo, seed in ((41120, gs.ALGO_PREFILL, 65), (65792, gs.ALGO_PREFILL_DENSE, 66)):
        Wb, B = layer(out, 256, 0.5, seed)
        p = packed(gs, Wb, B)
        xb = wl.random_activation_bits(T, 256, seed=seed + 7)
        y = to_bits(gs.linear(to_dev(xb), p, algo=algo))
        assert_within_bound(y, xb, Wb, B, tokens=sample_tokens(T, seed=seed), what=f"{out} rows algo {algo}")
    assert gs.device_status() == gs.GS_OK


def test_auto_dispatch_and_empty_batch(gs):
    import torch
    Wb, B = layer(1024, 1024, 0.5, 4)
    p = packed(gs, Wb, B)
    for T in (1, 16, 17, 24, 32, 33, 200):   # decode up to 16 tokens, tensor-core kernels from 17
        xb = wl.random_activation_bits(T, 1024, seed=T)
        assert_within_bound(to_bits(gs.linear(to_dev(xb), p)), xb, Wb, B, what=f"auto T={T}")
    x0 = torch.empty((0, 1024), dtype=torch.bfloat16, device="cuda")
    assert gs.linear(x0, p).shape == (0, 1024)


def test_deterministic_outputs(gs):
    Wb, B = layer(4096, 4096, 0.5, 6)
    p = packed(gs, Wb, B)
    for T, algo in ((16, gs.ALGO_DECODE), (1, gs.ALGO_DECODE), (300, gs.ALGO_PREFILL)):
        x = to_dev(wl.random_activation_bits(T, 4096, seed=5))
        a = to_bits(gs.linear(x, p, algo=algo))
        b = to_bits(gs.linear(x, p, algo=algo))
        assert np.array_equal(a, b)


def test_single_layer_workload(gs):
    """1024x1024 layer, exactly half of its 4096 groups kept, 8 tokens."""
    w = wl.workload(1)
    k = wl.keep_counts(w)
    Wb = wl.weight_bits(w, 0)
    B = wl.group_mask(w, 0, int(k[0]))
    xb = wl.activation_bits(w, 0, 8)
    p = packed(gs, Wb, B)
    assert p.kept == 2048
    for algo in (gs.ALGO_AUTO, gs.ALGO_DECODE, gs.ALGO_PREFILL):
        assert_within_bound(to_bits(gs.linear(to_dev(xb), p, algo=algo)), xb, Wb, B, what=f"cfg1 algo={algo}")


def test_block_workload_decode_batched(gs):
    """One LLaMA-2-7B-shaped block (7 projections, exactly 50 % of groups kept),
    decode with 1, 4 and 16 tokens, all layers in one batched launch."""
    import torch
    w = wl.workload(2)
    k = wl.keep_counts(w)
    Ws, Bs, ps = [], [], []
    for i in range(len(w.layers)):
        Wb = wl.weight_bits(w, i)
        B = wl.group_mask(w, i, int(k[i]))
        Ws.append(Wb)
        Bs.append(B)
        ps.append(packed(gs, Wb, B))
    assert sum(p.kept for p in ps) == w.budget
    for T in w.tokens:
        xs = [wl.activation_bits(w, i, T) for i in range(len(w.layers))]
        xd = [to_dev(x) for x in xs]
        ys = [torch.empty((T, L.out), dtype=torch.bfloat16, device="cuda") for L in w.layers]
        gs.linear_batched_into(xd, ps, ys)
        ys2 = [torch.empty_like(y) for y in ys]
        gs.linear_batched_into(xd, ps, ys2)
        for i in range(len(w.layers)):
            assert torch.equal(ys[i], ys2[i])          # deterministic for a fixed launch configuration
            assert_within_bound(to_bits(ys[i]), xs[i], Ws[i], Bs[i], what=f"cfg2 {w.layers[i].name} T={T}")
            # the single-layer call may split chunks differently (another fp32 order)
            y1 = gs.linear(xd[i], ps[i])
            assert_within_bound(to_bits(y1), xs[i], Ws[i], Bs[i], what=f"cfg2 single {w.layers[i].name} T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("n", [9, 12, 32])
def test_decode_batched_many_layers(gs, n):
    """More layers in one decode launch than the small parameter block holds
    (up to the 32-layer limit), with mixed shapes and densities, the split and
    unsplit unit paths, and T = 3 and 16."""
    import torch
    outs = [64, 200, 256, 512, 1000, 1024]
    inps = [256, 512, 1024, 2048, 2816]
    dens = [0.2, 0.5, 0.8, 1.0, 0.05]
    Ws, Bs, ps = [], [], []
    for i in range(n):
        out, inp, d = outs[i % len(outs)], inps[(3 * i) % len(inps)], dens[(5 * i) % len(dens)]
        Wb, B = layer(out, inp, d, 500 + i)
        Ws.append(Wb)
        Bs.append(B)
        ps.append(packed(gs, Wb, B))
    for T in (3, 16):
        xs = [wl.random_activation_bits(T, W.shape[1], seed=700 + 17 * i + T) for i, W in enumerate(Ws)]
        xd = [to_dev(x) for x in xs]
        ys = [torch.empty((T, W.shape[0]), dtype=torch.bfloat16, device="cuda") for W in Ws]
        gs.linear_batched_into(xd, ps, ys)
        for i in range(n):
            assert_within_bound(to_bits(ys[i]), xs[i], Ws[i], Bs[i], what=f"batched n={n} layer {i} T={T}")
    assert gs.device_status() == gs.GS_OK


@pytest.mark.parametrize("n,T", [(3, 200), (11, 300), (7, 1024)])   # T = 1024: the zero-filled kernel
def test_prefill_batched_matches_single(gs, n, T):
    """A batched prefill call (several layers with one T share launches of up
    to 8 layers) gives bit for bit the single-layer results and stays within
    the bound; layers without kept groups give zeros."""
    import torch
    shapes = [(4096, 4096, 0.5), (1000, 1024, 0.3), (512, 2816, 0.8), (300, 256, 0.0), (2048, 512, 1.0),
              (160, 768, 0.5), (1100, 2048, 0.05)]
    Ws, Bs, ps = [], [], []
    for i in range(n):
        out, inp, d = shapes[i % len(shapes)]
        Wb, B = layer(out, inp, d, 900 + i)
        Ws.append(Wb)
        Bs.append(B)
        ps.append(packed(gs, Wb, B))
    xs = [wl.random_activation_bits(T, W.shape[1], seed=950 + i) for i, W in enumerate(Ws)]
    xd = [to_dev(x) for x in xs]
    ys = [torch.full((T, W.shape[0]), 7.0, dtype=torch.bfloat16, device="cuda") for W in Ws]
    gs.linear_batched_into(xd, ps, ys)
    toks = sample_tokens(T, seed=n)
    for i in range(n):
        y1 = gs.linear(xd[i], ps[i])
        assert np.array_equal(to_bits(ys[i]), to_bits(y1)), f"layer {i}: batched != single"
        assert_within_bound(to_bits(ys[i]), xs[i], Ws[i], Bs[i], tokens=toks, what=f"batched prefill layer {i}")
    assert gs.device_status() == gs.GS_OK


def stack_blocks(w, k):
    """Blocks checked for a stack: the first, the last, and the blocks holding
    the sparsest and the densest layer of the layer-adaptive allocation."""
    groups = np.array([L.out * (L.inp // 256) for L in w.layers], dtype=np.float64)
    dens = np.asarray(k, dtype=np.float64) / groups
    nblk = len(w.layers) // 7
    return sorted({0, nblk - 1, int(np.argmin(dens)) // 7, int(np.argmax(dens)) // 7})


_stack_cache = {}


def stack_layer(gs, w, k, i):
    key = (w.cfg_id, w.variant, w.density, i)
    if key not in _stack_cache:
        _stack_cache.clear()                  # one layer resident at a time (the stacks are GBs)
        Wb = wl.weight_bits(w, i)
        B = wl.group_mask(w, i, int(k[i]))
        _stack_cache[key] = (Wb, B, packed(gs, Wb, B))
    return _stack_cache[key]


# (config, density, token counts): the full-size stacks of the 7B model with
# activation outliers at prefill, the 13B model over its token sweep, and the
# Qwen model over its density sweep at T = 1 and 1024.
STACK_CASES = [(3, 0.5, (2048,)), (4, 0.5, (1, 16, 128, 512, 2048)), (5, 0.3, (1, 1024)), (5, 0.5, (1, 1024)),
               (5, 0.7, (1, 1024))]


@pytest.mark.parametrize("cfg,d,Ts", STACK_CASES)
def test_stack_shapes_sampled(gs, cfg, d, Ts):
    """Every layer of the checked blocks of a full-size stack (first, last, and the
    blocks with the sparsest and densest layer), each at the config's token
    counts, checked on a deterministic token sample (all tokens when T <= 16)."""
    w = wl.workload(cfg, d)
    k = wl.keep_counts(w)
    assert int(k.sum()) == w.budget
    for b in stack_blocks(w, k):
        for i in range(7 * b, 7 * b + 7):
            Wb, B, p = stack_layer(gs, w, k, i)
            assert p.kept == int(k[i])
            for T in Ts:
                xb = wl.activation_bits(w, i, T)
                y = to_bits(gs.linear(to_dev(xb), p))
                assert_within_bound(y, xb, Wb, B, tokens=None if T <= 16 else sample_tokens(T, seed=i),
                                    what=f"cfg{cfg} d={d} {w.layers[i].name} T={T}")
    _stack_cache.clear()
    assert gs.device_status() == gs.GS_OK


def test_paper_allocation_blocks_batched(gs):
    """The paper-shaped allocation of the full 7B stack (Sec. 3.5 statistics): all
    seven projections of block 0 and of block 25 (Q/K near 8 %, down above 53 %) in
    one batched call per token count: T = 1 and 16 (decode, every token) and
    T = 2048 (prefill, token sample)."""
    import torch
    w = wl.workload(3, allocation="paper")
    k = wl.keep_counts(w)
    for b in (0, 25):
        ids = list(range(7 * b, 7 * b + 7))
        host = [(wl.weight_bits(w, i), wl.group_mask(w, i, int(k[i]))) for i in ids]
        ps = [packed(gs, Wb, B) for Wb, B in host]
        assert [p.kept for p in ps] == [int(k[i]) for i in ids]
        for T in (1, 16, 2048):
            xbs = [wl.activation_bits(w, i, T) for i in ids]
            ys = [torch.empty((T, w.layers[i].out), dtype=torch.bfloat16, device="cuda") for i in ids]
            gs.linear_batched_into([to_dev(xb) for xb in xbs], ps, ys)
            for j, i in enumerate(ids):
                Wb, B = host[j]
                assert_within_bound(to_bits(ys[j]), xbs[j], Wb, B,
                                    tokens=None if T <= 16 else sample_tokens(T, seed=i),
                                    what=f"paper allocation {w.layers[i].name} T={T}")
        del ps
    assert gs.device_status() == gs.GS_OK


def test_graph_capture_replay(gs):
    import torch
    Wb, B = layer(4096, 4096, 0.5, 6)
    p = packed(gs, Wb, B)
    for T, algo in ((16, gs.ALGO_DECODE), (256, gs.ALGO_PREFILL)):
        x = to_dev(wl.random_activation_bits(T, 4096, seed=T))
        y = torch.empty((T, 4096), dtype=torch.bfloat16, device="cuda")
        ref = to_bits(gs.linear(x, p, algo=algo))
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            gs.linear_into(x, p, y, algo=algo)   # warm-up outside capture
        torch.cuda.current_stream().wait_stream(s)
        g = torch.cuda.CUDAGraph()
        y.zero_()
        with torch.cuda.graph(g):
            gs.linear_into(x, p, y, algo=algo)
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(to_bits(y), ref)
