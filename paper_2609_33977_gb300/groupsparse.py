"""Python binding of libgroupsparse.so (argument marshalling only).

Every call goes straight to the C ABI declared in include/groupsparse.h; torch
is used for device memory and the current CUDA stream.  There is no fallback:
if the compiled library is missing or fails to load, importing this module
raises.
"""
from __future__ import annotations

import ctypes
from pathlib import Path
from typing import Optional, Sequence

import numpy as np
import torch

_PKG = Path(__file__).resolve().parent
LIB_PATH = _PKG / "libgroupsparse.so"

GS_OK, GS_ERR_INVALID_ARG, GS_ERR_UNSUPPORTED, GS_ERR_OOM, GS_ERR_CUDA, GS_ERR_DEVICE_TIMEOUT = range(6)
ALGO_AUTO, ALGO_DECODE, ALGO_PREFILL, ALGO_PREFILL_DENSE = 0, 1, 2, 3

_c_i64p = ctypes.POINTER(ctypes.c_int64)
_c_i32p = ctypes.POINTER(ctypes.c_int32)
_c_u16p = ctypes.POINTER(ctypes.c_uint16)


def _load(path: Path = LIB_PATH) -> ctypes.CDLL:
    if not path.exists():
        raise ImportError(f"{path} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(str(path))
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.gs_pack.argtypes = [vp, vp, i64, i64, i32, vp, ctypes.POINTER(vp)]
    lib.gs_pack_groups.argtypes = [vp, vp, i64, i64, i32, i32, vp, ctypes.POINTER(vp)]
    lib.gs_packed_group_shape.argtypes = [vp, _c_i32p, _c_i32p]
    lib.gs_linear.argtypes = [vp, vp, i64, vp, vp]
    lib.gs_linear_ex.argtypes = [vp, vp, i64, vp, vp, ctypes.c_int]
    lib.gs_linear_batched.argtypes = [i32, ctypes.POINTER(vp), ctypes.POINTER(vp), i64, ctypes.POINTER(vp), vp]
    lib.gs_unpack.argtypes = [vp, vp, vp]
    lib.gs_select_groups.argtypes = [vp, i64, vp, vp, vp]
    lib.gs_packed_info.argtypes = [vp, _c_i64p, _c_i64p, _c_i64p, ctypes.POINTER(ctypes.c_size_t)]
    lib.gs_packed_export.argtypes = [vp, _c_i64p, _c_i32p, _c_u16p, _c_i32p, _c_u16p]
    lib.gs_free.argtypes = [vp]
    lib.gs_free.restype = None
    lib.gs_status_string.argtypes = [ctypes.c_int]
    lib.gs_status_string.restype = ctypes.c_char_p
    lib.gs_device_status.argtypes = [vp]
    lib.gs_launch_count.argtypes = []
    lib.gs_launch_count.restype = ctypes.c_int64
    lib.gs_preserved_rates.argtypes = [i32, vp, vp, vp, i64, vp, vp, i32, vp, vp]
    lib.gs_gumbel_select.argtypes = [vp, vp, i64, ctypes.c_float, vp, vp, vp, vp]
    lib.gs_masked_linear_backward_workspace.argtypes = [vp, i32, ctypes.POINTER(ctypes.c_size_t)]
    lib.gs_masked_linear_backward.argtypes = [vp, vp, vp, vp, i64, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.gs_debug_fail_alloc.argtypes = [i64]
    lib.gs_debug_inject_wait.argtypes = [ctypes.c_int, ctypes.c_uint64]
    for fn in (lib.gs_pack, lib.gs_linear, lib.gs_linear_ex, lib.gs_linear_batched, lib.gs_unpack,
               lib.gs_packed_info, lib.gs_packed_export, lib.gs_device_status, lib.gs_select_groups,
               lib.gs_preserved_rates, lib.gs_debug_fail_alloc, lib.gs_debug_inject_wait, lib.gs_pack_groups,
               lib.gs_packed_group_shape, lib.gs_gumbel_select, lib.gs_masked_linear_backward_workspace,
               lib.gs_masked_linear_backward):
        fn.restype = ctypes.c_int
    return lib


lib = _load()


class GroupSparseError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {lib.gs_status_string(status).decode()} (status {status})")
        self.status = status


def _check(status: int, what: str) -> None:
    if status != GS_OK:
        raise GroupSparseError(status, what)


def _stream_ptr(stream: Optional[torch.cuda.Stream] = None) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _require_cuda(t: torch.Tensor, dtype: torch.dtype, name: str) -> None:
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


class Packed:
    """A packed group-sparse weight (owns the library handle)."""

    def __init__(self, handle: int, out: int, inp: int, g_out: int = 1, g_in: int = 256):
        self._h = ctypes.c_void_p(handle)
        self.out = out
        self.inp = inp
        self.g_out = g_out
        self.g_in = g_in

    @property
    def handle(self) -> ctypes.c_void_p:
        if not self._h:
            raise ValueError("packed weight already freed")
        return self._h

    @property
    def G(self) -> int:
        return self.inp // self.g_in

    def info(self):
        out, inp, kept = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        nbytes = ctypes.c_size_t()
        _check(lib.gs_packed_info(self.handle, ctypes.byref(out), ctypes.byref(inp), ctypes.byref(kept),
                                  ctypes.byref(nbytes)), "gs_packed_info")
        return {"out": out.value, "in": inp.value, "kept": kept.value, "device_bytes": nbytes.value}

    @property
    def kept(self) -> int:
        return self.info()["kept"]

    def export(self):
        """Host copies of the packed layout: offsets, row_idx, tiles, win_off16, kmask16
        (square groups: offsets, row_idx = block rows, tiles [K, g, g])."""
        K = self.kept
        G = self.G
        if self.g_out > 1:
            offsets = np.zeros(G + 1, np.int64)
            rows = np.zeros(max(K, 1), np.int32)
            tiles = np.zeros((max(K, 1), self.g_out, self.g_in), np.uint16)
            _check(lib.gs_packed_export(self.handle, offsets.ctypes.data_as(_c_i64p), rows.ctypes.data_as(_c_i32p),
                                        tiles.ctypes.data_as(_c_u16p), None, None), "gs_packed_export")
            return {"offsets": offsets, "row_idx": rows[:K], "tiles": tiles[:K]}
        nw16 = (self.out + 15) // 16
        offsets = np.zeros(G + 1, np.int64)
        row_idx = np.zeros(max(K, 1), np.int32)
        tiles = np.zeros((max(K, 1), self.g_in), np.uint16)
        win = np.zeros((G, nw16 + 1), np.int32)
        km = np.zeros((G, nw16), np.uint16)
        _check(lib.gs_packed_export(self.handle, offsets.ctypes.data_as(_c_i64p), row_idx.ctypes.data_as(_c_i32p),
                                    tiles.ctypes.data_as(_c_u16p), win.ctypes.data_as(_c_i32p),
                                    km.ctypes.data_as(_c_u16p)), "gs_packed_export")
        return {"offsets": offsets, "row_idx": row_idx[:K], "tiles": tiles[:K], "win_off16": win, "kmask16": km}

    def free(self) -> None:
        if self._h:
            lib.gs_free(self._h)
            self._h = ctypes.c_void_p(None)

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def pack(W: torch.Tensor, mask: torch.Tensor, stream: Optional[torch.cuda.Stream] = None) -> Packed:
    """Pack a bf16 weight [out, in] with a uint8/bool group mask [out, in/256] (nonzero = keep)."""
    _require_cuda(W, torch.bfloat16, "W")
    if mask.dtype == torch.bool:
        mask = mask.to(torch.uint8)
    _require_cuda(mask, torch.uint8, "mask")
    out, inp = W.shape
    if tuple(mask.shape) != (out, inp // 256):
        raise ValueError("mask must be [out, in/256]")
    h = ctypes.c_void_p()
    _check(lib.gs_pack(W.data_ptr(), mask.data_ptr(), out, inp, 256, _stream_ptr(stream), ctypes.byref(h)),
           "gs_pack")
    return Packed(h.value, out, inp)


def pack_groups(W: torch.Tensor, mask: torch.Tensor, g_out: int, g_in: int,
                stream: Optional[torch.cuda.Stream] = None) -> Packed:
    """Pack a bf16 weight [out, in] with a group mask [out/g_out, in/g_in] (nonzero = keep)
    for g_out x g_in groups: (1, 256), (1, 128) or square g x g, g in {16, 32, 64, 128}."""
    _require_cuda(W, torch.bfloat16, "W")
    if mask.dtype == torch.bool:
        mask = mask.to(torch.uint8)
    _require_cuda(mask, torch.uint8, "mask")
    out, inp = W.shape
    if out % g_out or inp % g_in or tuple(mask.shape) != (out // g_out, inp // g_in):
        raise ValueError("mask must be [out/g_out, in/g_in] and the groups must tile W")
    h = ctypes.c_void_p()
    _check(lib.gs_pack_groups(W.data_ptr(), mask.data_ptr(), out, inp, g_out, g_in, _stream_ptr(stream),
                              ctypes.byref(h)), "gs_pack_groups")
    return Packed(h.value, out, inp, g_out, g_in)


def linear_into(x: torch.Tensor, p: Packed, y: torch.Tensor, algo: int = ALGO_AUTO,
                stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    _require_cuda(x, torch.bfloat16, "x")
    _require_cuda(y, torch.bfloat16, "y")
    T = x.shape[0]
    if x.dim() != 2 or x.shape[1] != p.inp or tuple(y.shape) != (T, p.out):
        raise ValueError("x must be [T, in] and y [T, out]")
    _check(lib.gs_linear_ex(x.data_ptr(), p.handle, T, y.data_ptr(), _stream_ptr(stream), algo), "gs_linear")
    return y


def linear(x: torch.Tensor, p: Packed, algo: int = ALGO_AUTO, stream: Optional[torch.cuda.Stream] = None):
    """y = x (W (.) M)^T as bf16 [T, out]."""
    y = torch.empty((x.shape[0], p.out), dtype=torch.bfloat16, device=x.device)
    return linear_into(x, p, y, algo, stream)


def linear_batched_into(xs: Sequence[torch.Tensor], ps: Sequence[Packed], ys: Sequence[torch.Tensor],
                        stream: Optional[torch.cuda.Stream] = None) -> None:
    n = len(ps)
    if not (len(xs) == len(ys) == n):
        raise ValueError("xs, ps, ys must have the same length")
    if n == 0:
        return
    T = xs[0].shape[0]
    for x, p, y in zip(xs, ps, ys):
        _require_cuda(x, torch.bfloat16, "x")
        _require_cuda(y, torch.bfloat16, "y")
        if x.shape[0] != T or x.shape[1] != p.inp or tuple(y.shape) != (T, p.out):
            raise ValueError("every x must be [T, in_i] and y [T, out_i] with one T")
    arr = ctypes.c_void_p * n
    xa = arr(*[x.data_ptr() for x in xs])
    pa = arr(*[p.handle.value for p in ps])
    ya = arr(*[y.data_ptr() for y in ys])
    _check(lib.gs_linear_batched(n, xa, pa, T, ya, _stream_ptr(stream)), "gs_linear_batched")


def unpack(p: Packed, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """W_hat = W (.) M as bf16 [out, in]; pruned groups are +0.0."""
    W = torch.empty((p.out, p.inp), dtype=torch.bfloat16, device="cuda")
    _check(lib.gs_unpack(p.handle, W.data_ptr(), _stream_ptr(stream)), "gs_unpack")
    return W


def select_groups(logits: torch.Tensor, mask: Optional[torch.Tensor] = None,
                  kept: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
    """Selector export (Sec. 2.2; App. F): mask = [sigmoid(logits) > 1/2] as uint8 0/1 of
    the logits' shape, and kept = the number of ones as an int64 [1] device tensor.
    For one layer with 1x256 groups, logits are float32 [out, in/256]."""
    _require_cuda(logits, torch.float32, "logits")
    if mask is None:
        mask = torch.empty(logits.shape, dtype=torch.uint8, device=logits.device)
    else:
        _require_cuda(mask, torch.uint8, "mask")
        if mask.numel() != logits.numel():
            raise ValueError("mask must hold one byte per logit")
    if kept is None:
        kept = torch.empty((1,), dtype=torch.int64, device=logits.device)
    else:
        _require_cuda(kept, torch.int64, "kept")
        if kept.numel() < 1:
            raise ValueError("kept must hold at least one int64")
    _check(lib.gs_select_groups(logits.data_ptr(), logits.numel(), mask.data_ptr(), kept.data_ptr(),
                                _stream_ptr(stream)), "gs_select_groups")
    return mask, kept


def pack_from_logits(W: torch.Tensor, logits: torch.Tensor,
                     stream: Optional[torch.cuda.Stream] = None) -> Packed:
    """Export a layer's selectors from its float32 logits [out, in/256] and pack W with them."""
    mask, _ = select_groups(logits, stream=stream)
    return pack(W, mask, stream)


_QKV = {"q": "q", "k": "k", "v": "v", "q_proj": "q", "k_proj": "k", "v_proj": "v"}


def preserved_report(kept: Sequence[int], shapes: Sequence[Sequence[int]],
                     names: Optional[Sequence[str]] = None, group: int = 256) -> dict:
    """Preserved rates of exported masks (App. F) from per-layer kept-group counts,
    computed by gs_preserved_rates: each layer's active over total weights, the
    global rate (1 - s of Eq. 2) and, for layers named q, k and v (or q_proj,
    k_proj, v_proj) under one dotted prefix, the mean of the three, keyed by
    that prefix.  This function only arranges the arguments."""
    if len(kept) != len(shapes) or (names is not None and len(names) != len(kept)):
        raise ValueError("kept, shapes (and names) must have the same length")
    names = list(names) if names is not None else [str(i) for i in range(len(kept))]
    n = len(kept)
    k_arr = np.ascontiguousarray(kept, dtype=np.int64)
    sh = np.asarray(shapes, dtype=np.int64).reshape(n, 2)
    d_out = np.ascontiguousarray(sh[:, 0])
    d_in = np.ascontiguousarray(sh[:, 1])
    index = {m: i for i, m in enumerate(names)}
    prefixes, triples = [], []
    for m in names:
        prefix, _, last = m.rpartition(".")
        if _QKV.get(last) != "q":
            continue
        trio = {}
        for m2 in names:
            p2, _, l2 = m2.rpartition(".")
            if p2 == prefix and l2 in _QKV:
                trio[_QKV[l2]] = index[m2]
        if len(trio) == 3:
            prefixes.append(prefix)
            triples.append((trio["q"], trio["k"], trio["v"]))
    qkv_idx = np.ascontiguousarray(np.asarray(triples, dtype=np.int32).reshape(-1, 3))
    rates = np.zeros(max(n, 1), np.float64)
    qkv_rates = np.zeros(max(len(triples), 1), np.float64)
    glob = ctypes.c_double()
    _check(lib.gs_preserved_rates(n, k_arr.ctypes.data, d_out.ctypes.data, d_in.ctypes.data, int(group),
                                  rates.ctypes.data, ctypes.byref(glob), len(triples), qkv_idx.ctypes.data,
                                  qkv_rates.ctypes.data), "gs_preserved_rates")
    return {"layers": {m: float(rates[i]) for i, m in enumerate(names)}, "global": glob.value,
            "qkv": {pf: float(qkv_rates[j]) for j, pf in enumerate(prefixes)}}


def gumbel_select(logits: torch.Tensor, noise: torch.Tensor, tau: float,
                  stream: Optional[torch.cuda.Stream] = None):
    """One Gumbel-Sigmoid sample of the selectors (Sec. 2.2): mask = [l + L > 0] (uint8),
    dsdl = d sigmoid((l + L) / tau) / dl (float32, the straight-through derivative) and the
    kept count (int64 [1]); L is the caller's logistic noise, of the logits' shape."""
    _require_cuda(logits, torch.float32, "logits")
    _require_cuda(noise, torch.float32, "noise")
    if noise.shape != logits.shape:
        raise ValueError("noise must have the logits' shape")
    mask = torch.empty(logits.shape, dtype=torch.uint8, device=logits.device)
    dsdl = torch.empty(logits.shape, dtype=torch.float32, device=logits.device)
    kept = torch.empty((1,), dtype=torch.int64, device=logits.device)
    _check(lib.gs_gumbel_select(logits.data_ptr(), noise.data_ptr(), logits.numel(), float(tau), mask.data_ptr(),
                                dsdl.data_ptr(), kept.data_ptr(), _stream_ptr(stream)), "gs_gumbel_select")
    return mask, dsdl, kept


def masked_linear_backward(x: torch.Tensor, W: torch.Tensor, p: Packed, dy: torch.Tensor, dsdl: torch.Tensor,
                           want_dx: bool = True, stream: Optional[torch.cuda.Stream] = None):
    """Straight-through backward of y = x W_hat^T (Sec. 2.2): (dlogits float32 of the
    mask's shape, dx bf16 [T, in] or None).  p is W packed with the sampled mask."""
    _require_cuda(x, torch.bfloat16, "x")
    _require_cuda(W, torch.bfloat16, "W")
    _require_cuda(dy, torch.bfloat16, "dy")
    _require_cuda(dsdl, torch.float32, "dsdl")
    T = x.shape[0]
    if tuple(W.shape) != (p.out, p.inp) or x.shape[1] != p.inp or tuple(dy.shape) != (T, p.out):
        raise ValueError("W must be [out, in], x [T, in] and dy [T, out]")
    shape = (p.out // p.g_out, p.inp // p.g_in)
    if tuple(dsdl.shape) != shape:
        raise ValueError(f"dsdl must be {shape}")
    nbytes = ctypes.c_size_t()
    _check(lib.gs_masked_linear_backward_workspace(p.handle, 1 if want_dx else 0, ctypes.byref(nbytes)),
           "gs_masked_linear_backward_workspace")
    ws = torch.empty((nbytes.value,), dtype=torch.uint8, device=x.device)
    dl = torch.empty(shape, dtype=torch.float32, device=x.device)
    dx = torch.empty((T, p.inp), dtype=torch.bfloat16, device=x.device) if want_dx else None
    _check(lib.gs_masked_linear_backward(x.data_ptr(), W.data_ptr(), p.handle, dy.data_ptr(), T, dsdl.data_ptr(),
                                         dl.data_ptr(), dx.data_ptr() if dx is not None else None,
                                         ws.data_ptr(), nbytes.value, _stream_ptr(stream)),
           "gs_masked_linear_backward")
    return dl, dx


def debug_fail_alloc(nth: int) -> None:
    """Test hook: the nth device allocation the library makes from now on fails (0 disarms)."""
    _check(lib.gs_debug_fail_alloc(int(nth)), "gs_debug_fail_alloc")


def debug_inject_wait(algo: int, limit_ns: int) -> None:
    """Test hook: the next launch of that kernel family times out on a word nothing sets."""
    _check(lib.gs_debug_inject_wait(int(algo), int(limit_ns)), "gs_debug_inject_wait")


def device_status(stream: Optional[torch.cuda.Stream] = None) -> int:
    return int(lib.gs_device_status(_stream_ptr(stream)))


def launch_count() -> int:
    return int(lib.gs_launch_count())
