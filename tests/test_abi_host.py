"""The C-ABI library loads, exports every symbol include/*.h declares, and rejects
bad arguments on the host before touching any device (no GPU needed)."""
import ctypes
import re
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parent.parent


def declared_functions():
    names = set()
    for h in (ROOT / "include").glob("*.h"):
        text = re.sub(r"/\*.*?\*/", "", h.read_text(), flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(gs_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def lib(built_lib):
    return ctypes.CDLL(str(built_lib))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("gs_pack", "gs_linear", "gs_unpack", "gs_free", "gs_packed_info", "gs_status_string"):
        assert required in names
    assert len(names) >= 10


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_loads(built_lib):
    from paper_2609_33977_gb300 import groupsparse as gs
    assert gs.lib.gs_status_string(0) == b"ok"
    assert gs.lib.gs_status_string(5) == b"device wait timed out"


def test_host_side_validation(lib):
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.gs_pack.argtypes = [vp, vp, i64, i64, i32, vp, ctypes.POINTER(vp)]
    lib.gs_linear.argtypes = [vp, vp, i64, vp, vp]
    lib.gs_linear_ex.argtypes = [vp, vp, i64, vp, vp, ctypes.c_int]
    lib.gs_unpack.argtypes = [vp, vp, vp]
    lib.gs_linear_batched.argtypes = [i32, vp, vp, i64, vp, vp]
    lib.gs_packed_info.argtypes = [vp, vp, vp, vp, vp]
    lib.gs_packed_export.argtypes = [vp, vp, vp, vp, vp, vp]
    lib.gs_select_groups.argtypes = [vp, i64, vp, vp, vp]
    lib.gs_free.argtypes = [vp]
    lib.gs_free.restype = None
    h = vp(12345)
    fake = 0x10000  # never dereferenced: each call below fails validation first
    INVALID, UNSUPPORTED = 1, 2
    assert lib.gs_pack(None, fake, 4, 256, 256, None, ctypes.byref(h)) == INVALID
    assert h.value is None                                            # handle cleared on failure
    assert lib.gs_pack(fake, None, 4, 256, 256, None, ctypes.byref(h)) == INVALID
    assert lib.gs_pack(fake, fake, 4, 256, 256, None, None) == INVALID
    assert lib.gs_pack(fake, fake, 0, 256, 256, None, ctypes.byref(h)) == INVALID
    assert lib.gs_pack(fake, fake, 4, 300, 256, None, ctypes.byref(h)) == INVALID   # in % 256 != 0
    assert lib.gs_pack(fake, fake, 4, 256, 128, None, ctypes.byref(h)) == UNSUPPORTED
    assert lib.gs_pack(fake + 2, fake, 4, 256, 256, None, ctypes.byref(h)) == INVALID  # misaligned W
    assert lib.gs_linear(fake, None, 4, fake, None) == INVALID
    assert lib.gs_linear_ex(fake, None, 4, fake, None, 7) == INVALID
    assert lib.gs_unpack(None, fake, None) == INVALID
    assert lib.gs_linear_batched(-1, None, None, 1, None, None) == INVALID
    assert lib.gs_linear_batched(33, fake, fake, 1, fake, None) == INVALID
    assert lib.gs_linear_batched(0, None, None, 1, None, None) == 0
    assert lib.gs_packed_info(None, None, None, None, None) == INVALID
    assert lib.gs_packed_export(None, None, None, None, None, None) == INVALID
    assert lib.gs_select_groups(fake, -1, fake + 0x1000, None, None) == INVALID
    assert lib.gs_select_groups(fake, 1 << 36, fake + 0x1000, None, None) == INVALID
    assert lib.gs_select_groups(None, 8, fake, None, None) == INVALID
    assert lib.gs_select_groups(fake, 8, None, None, None) == INVALID
    assert lib.gs_select_groups(fake + 4, 8, fake + 0x1000, None, None) == INVALID   # misaligned logits
    assert lib.gs_select_groups(fake, 8, fake + 0x1008, None, None) == INVALID       # misaligned mask
    assert lib.gs_select_groups(fake, 8, fake + 0x1000, fake + 4, None) == INVALID   # misaligned count
    assert lib.gs_select_groups(fake, 8, fake + 16, None, None) == INVALID           # mask overlaps logits
    assert lib.gs_select_groups(None, 0, None, None, None) == 0                      # empty: nothing to do
    lib.gs_pack_index_noalloc.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    m, o, w, k = 0x100000, 0x200000, 0x300000, 0x400000   # mask, offsets, window offsets, window masks
    assert lib.gs_pack_index_noalloc(m, 16, 512, o + 4, w, k, None) == INVALID     # int64 offsets at 4 B
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w + 2, k, None) == INVALID     # int32 offsets at 2 B
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w, k + 1, None) == INVALID     # uint16 masks at 1 B
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, o + 16, k, None) == INVALID    # outputs overlap
    assert lib.gs_pack_index_noalloc(m, 16, 512, o, w, m + 16, None) == INVALID    # output overlaps the mask
    assert lib.gs_pack_index_noalloc(None, 16, 512, o, w, k, None) == INVALID
    assert lib.gs_pack_index_noalloc(m, 16, 300, o, w, k, None) == INVALID
    lib.gs_free(None)


def test_header_is_plain_c(tmp_path):
    # the boundary is a C ABI: the header compiles as strict C99 (no C++ or torch types) and as C++
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "use_header.c"
    src.write_text('#include "groupsparse.h"\n'
                   "int main(void) { gs_packed* p = 0; (void)p; return gs_status_string(GS_OK)[0] == 0; }\n")
    for cmd in ([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror"],
                [gcc, "-x", "c++", "-std=c++17", "-Wall", "-Wextra", "-Werror"]):
        r = subprocess.run(cmd + [f"-I{ROOT / 'include'}", "-fsyntax-only", str(src)], capture_output=True, text=True)
        assert r.returncode == 0, r.stderr


def test_preserved_rates_call(lib):
    # App. F arithmetic lives in the library (host only, no device work):
    # exact per-layer rates, the Eq. 2 global rate and the Q/K/V plain mean
    import numpy as np
    from oracle import groupsparse_oracle as orc
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    lib.gs_preserved_rates.argtypes = [i32, vp, vp, vp, i64, vp, vp, i32, vp, vp]
    rng = np.random.default_rng(11)
    shapes = [(48, 512), (16, 512), (16, 512), (32, 768), (64, 1024)]
    Bs = [(rng.random((o, i // 256)) < 0.45).astype(np.uint8) for o, i in shapes]
    kept = np.array([int(B.sum()) for B in Bs], np.int64)
    d_out = np.array([s[0] for s in shapes], np.int64)
    d_in = np.array([s[1] for s in shapes], np.int64)
    qkv = np.array([[0, 1, 2], [2, 1, 0]], np.int32)
    rates = np.zeros(5)
    qrates = np.zeros(2)
    glob = ctypes.c_double()
    assert lib.gs_preserved_rates(5, kept.ctypes.data, d_out.ctypes.data, d_in.ctypes.data, 256, rates.ctypes.data,
                                  ctypes.byref(glob), 2, qkv.ctypes.data, qrates.ctypes.data) == 0
    for i, B in enumerate(Bs):
        assert rates[i] == orc.preserved_rate(B)
    assert glob.value == pytest.approx(orc.global_preserved_rate(Bs, shapes), abs=1e-15)
    assert qrates[0] == pytest.approx(orc.qkv_preserved_rate(Bs[0], Bs[1], Bs[2]), abs=1e-15)
    assert qrates[1] == pytest.approx(orc.qkv_preserved_rate(Bs[2], Bs[1], Bs[0]), abs=1e-15)
    INVALID = 1
    bad = kept.copy()
    bad[3] = 32 * 3 + 1                      # more kept groups than the layer holds
    assert lib.gs_preserved_rates(5, bad.ctypes.data, d_out.ctypes.data, d_in.ctypes.data, 256, None, None, 0,
                                  None, None) == INVALID
    neg = np.array([[0, 1, 5]], np.int32)    # index out of range
    assert lib.gs_preserved_rates(5, kept.ctypes.data, d_out.ctypes.data, d_in.ctypes.data, 256, None, None, 1,
                                  neg.ctypes.data, qrates.ctypes.data) == INVALID
    assert lib.gs_preserved_rates(1, None, d_out.ctypes.data, d_in.ctypes.data, 256, None, None, 0, None,
                                  None) == INVALID
    assert lib.gs_preserved_rates(0, None, None, None, 256, None, ctypes.byref(glob), 0, None, None) == 0
    assert glob.value == 0.0


def test_debug_hooks_validate_arguments(lib):
    lib.gs_debug_fail_alloc.argtypes = [ctypes.c_int64]
    lib.gs_debug_inject_wait.argtypes = [ctypes.c_int, ctypes.c_uint64]
    INVALID = 1
    assert lib.gs_debug_fail_alloc(-1) == INVALID
    assert lib.gs_debug_fail_alloc(0) == 0
    assert lib.gs_debug_inject_wait(0, 1000) == INVALID          # AUTO is not a kernel family
    assert lib.gs_debug_inject_wait(1, 2_000_000_000) == INVALID  # above 1 s
    assert lib.gs_debug_inject_wait(1, 0) == 0 and lib.gs_debug_inject_wait(2, 0) == 0
    assert lib.gs_debug_inject_wait(3, 0) == 0                 # the zero-filled prefill kernel
    assert lib.gs_debug_inject_wait(4, 1000) == INVALID        # no such family
