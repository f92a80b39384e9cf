"""Host-only checks of the C ABI: the library loads, exports every symbol that
include/slim.h declares, sizes workspaces, and rejects bad arguments before
anything is enqueued (these calls never reach a CUDA launch)."""
import ctypes
import os
import re

import pytest

from paper_2012_11346_gb300 import slim

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in sorted(os.listdir(os.path.join(ROOT, "include")))
           if f.endswith(".h")]

OK, INVALID, UNSUPPORTED, WORKSPACE = 0, 1, 2, 3


def declared_symbols():
    names = set()
    for h in HEADERS:
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names.update(re.findall(r"\b(slim_[a-z0-9_]+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(slim._LIB_PATH):
        from paper_2012_11346_gb300 import build
        build.build()
    return slim.library()


def test_every_declared_symbol_is_exported(lib):
    names = declared_symbols()
    assert "slim_fwd" in names and "slim_bwd" in names
    for n in names:
        assert hasattr(lib, n), n
        assert n in slim.SIGNATURES, f"binding lacks {n}"


def test_status_strings(lib):
    for code, name in slim.STATUS.items():
        assert slim.status_string(code).startswith(name)
    assert lib.slim_version() >= 100


def ws(B, H, L, d, M, C, dt=0, ft=0, bwd=False):
    n = ctypes.c_size_t(0)
    fn = slim.library().slim_bwd_workspace_size if bwd else slim.library().slim_fwd_workspace_size
    st = fn(B, H, L, d, M, C, dt, ft, ctypes.byref(n))
    return st, n.value


def test_workspace_sizes_scale_with_C_not_L(lib):
    for bwd in (False, True):
        st, a = ws(2, 8, 32768, 64, 256, 64, 1, 0, bwd)
        assert st == OK and a > 0
        _, b = ws(2, 8, 32768, 64, 256, 4096, 1, 0, bwd)
        _, c = ws(2, 8, 65536, 64, 256, 4096, 1, 0, bwd)
        assert b > a and c == b                    # O(C), independent of L
        _, big = ws(2, 8, 32768, 64, 256, 32768, 1, 0, bwd)
        _, half = ws(2, 8, 32768, 64, 256, 16384, 1, 0, bwd)
        assert 1.8 < big / half < 2.1              # linear in C
        _, clamp = ws(2, 8, 1000, 64, 256, 5000, 1, 0, bwd)
        _, same = ws(2, 8, 1000, 64, 256, 1000, 1, 0, bwd)
        assert clamp == same                       # C > L behaves as C = L


@pytest.mark.parametrize("args,code", [
    ((0, 1, 8, 16, 32, 4), INVALID),     # B < 1
    ((1, 0, 8, 16, 32, 4), INVALID),     # H < 1
    ((1, 1, -1, 16, 32, 4), INVALID),    # L < 0
    ((1, 1, 8, 16, 32, 0), INVALID),     # C < 1
    ((1, 1, 8, 48, 32, 4), UNSUPPORTED),  # d not in {16, 32, 64, 128}
    ((1, 1, 8, 16, 24, 4), UNSUPPORTED),  # M not a multiple of 16
    ((1, 1, 8, 16, 272, 4), UNSUPPORTED),  # M > 256
])
def test_workspace_size_rejects(lib, args, code):
    assert ws(*args)[0] == code
    assert ws(*args, bwd=True)[0] == code


def test_bad_enums_and_null_out(lib):
    n = ctypes.c_size_t(0)
    assert lib.slim_fwd_workspace_size(1, 1, 8, 16, 32, 4, 7, 0, ctypes.byref(n)) == INVALID
    assert lib.slim_fwd_workspace_size(1, 1, 8, 16, 32, 4, 0, 9, ctypes.byref(n)) == INVALID
    assert lib.slim_fwd_workspace_size(1, 1, 8, 16, 32, 4, 0, 0, None) == INVALID


FAKE = 0x10000  # aligned, never dereferenced: every call below fails validation first


def fwd_call(lib, ptrs=None, dims=(1, 1, 8, 16, 32, 4), dt=0, ft=0, wsp=FAKE, wsb=0, lo=(None, None)):
    p = ptrs or [FAKE] * 7
    return lib.slim_fwd(p[0], p[1], p[2], p[3], *dims, dt, ft, p[4], p[5], p[6], lo[0], lo[1],
                        wsp, wsb, None)


def bwd_call(lib, ptrs=None, dims=(1, 1, 8, 16, 32, 4), wsp=FAKE, wsb=0, lo=(None, None)):
    p = ptrs or [FAKE] * 12
    return lib.slim_bwd(*p[:8], lo[0], lo[1], *dims, 0, 0, *p[8:12], wsp, wsb, None)


def test_fwd_rejects_before_launch(lib):
    for i in range(7):
        ptrs = [FAKE] * 7
        ptrs[i] = None
        assert fwd_call(lib, ptrs) == INVALID
        ptrs[i] = FAKE + 8                      # not 16-byte aligned
        assert fwd_call(lib, ptrs) == INVALID
    assert fwd_call(lib, dims=(1, 1, 8, 16, 32, 0)) == INVALID
    assert fwd_call(lib, dims=(1, 1, 8, 20, 32, 4)) == UNSUPPORTED
    _, need = ws(1, 1, 8, 16, 32, 4)
    assert fwd_call(lib, wsb=need - 1) == WORKSPACE
    assert fwd_call(lib, wsp=None, wsb=need) == WORKSPACE
    assert fwd_call(lib, wsp=FAKE + 16, wsb=need) == INVALID   # workspace not 256-aligned
    assert fwd_call(lib, lo=(FAKE + 4, None)) == INVALID         # misaligned residual
    assert fwd_call(lib, lo=(None, FAKE + 8), wsb=need - 1) == INVALID


def test_bwd_rejects_before_launch(lib):
    for i in range(12):
        ptrs = [FAKE] * 12
        ptrs[i] = None
        assert bwd_call(lib, ptrs) == INVALID
        ptrs[i] = FAKE + 4
        assert bwd_call(lib, ptrs) == INVALID
    _, need = ws(1, 1, 8, 16, 32, 4, bwd=True)
    assert bwd_call(lib, wsb=need - 1) == WORKSPACE
    assert bwd_call(lib, dims=(1, 1, 8, 16, 31, 4)) == UNSUPPORTED
    assert bwd_call(lib, lo=(FAKE, FAKE + 4)) == INVALID


def test_binding_refuses_cpu_tensors():
    import torch
    x = torch.zeros(1, 1, 8, 16)
    with pytest.raises(RuntimeError):
        slim.forward(x, x, x, torch.zeros(32, 16), 4)


def test_bwd_schedule_arguments(lib):
    n, ring = ctypes.c_int(-1), ctypes.c_int(-1)
    # count only (no buffer), then the tensor-core problems it serves
    assert lib.slim_bwd_schedule(8, 8, 4096, 64, 256, 1024, 1, 0, None, 0, ctypes.byref(n),
                                 ctypes.byref(ring)) == OK
    assert n.value == 4 * 64 * 8 + 64 + 16 and ring.value == 2
    buf = (ctypes.c_int * 6)()
    assert lib.slim_bwd_schedule(8, 8, 4096, 64, 256, 1024, 1, 0, buf, 2, ctypes.byref(n),
                                 None) == OK
    assert list(buf) == [0, 3, 0, 0, 3, 1]  # the first two tickets: tiles of the last slice
    # argument errors before anything else
    assert lib.slim_bwd_schedule(8, 8, 4096, 64, 256, 1024, 1, 0, None, 0, None, None) == INVALID
    assert lib.slim_bwd_schedule(8, 8, 4096, 64, 256, 1024, 1, 0, None, 4, ctypes.byref(n),
                                 None) == INVALID
    assert lib.slim_bwd_schedule(8, 8, 4096, 64, 256, 0, 1, 0, None, 0, ctypes.byref(n),
                                 None) == INVALID
    # problems the tensor-core kernels do not take: fp32, d = 128, slices under 64 rows
    for args in ((4, 12, 8192, 64, 128, 512, 0, 1), (1, 4, 65536, 128, 256, 16, 1, 0),
                 (2, 8, 32768, 64, 256, 16, 1, 0)):
        assert lib.slim_bwd_schedule(*args, None, 0, ctypes.byref(n), None) == UNSUPPORTED


SQUARE = 2


def test_square_map_needs_M_equal_d(lib):
    assert ws(1, 1, 8, 16, 16, 4, 0, SQUARE)[0] == OK
    assert ws(1, 1, 8, 16, 32, 4, 0, SQUARE)[0] == INVALID      # g(x)_i = x_i^2 has M = d
    assert ws(1, 1, 8, 64, 64, 4, 1, SQUARE, bwd=True)[0] == OK
    n = ctypes.c_int(-1)
    # the quadratic map runs on the fp32-compute kernels
    assert lib.slim_path_for(8, 8, 4096, 64, 64, 1024, 1, SQUARE, ctypes.byref(n)) == OK
    assert n.value == 0


def test_omega_optional_only_for_square(lib):
    _, need = ws(1, 1, 8, 16, 16, 4, 0, SQUARE)
    p = [FAKE] * 7
    p[3] = None                                                   # no Omega
    assert fwd_call(lib, p, dims=(1, 1, 8, 16, 32, 4), ft=0) == INVALID
    # with the quadratic map a null Omega passes validation; a too-small
    # workspace is then the first error
    assert fwd_call(lib, p, dims=(1, 1, 8, 16, 16, 4), ft=SQUARE, wsb=need - 1) == WORKSPACE


def fwd_from_call(lib, init, dims=(1, 1, 8, 16, 32, 4), wsb=0):
    p = [FAKE] * 7
    return lib.slim_fwd_from(p[0], p[1], p[2], p[3], *dims, 0, 0, *init, p[4], p[5], p[6], None,
                             None, FAKE, wsb, None)


def bwd_from_call(lib, gin, gout, dims=(1, 1, 8, 16, 32, 4), wsb=0):
    p = [FAKE] * 12
    return lib.slim_bwd_from(*p[:8], None, None, gin[0], gin[1], *dims, 0, 0, *p[8:12], gout[0],
                             gout[1], FAKE, wsb, None)


def test_streaming_arguments_rejected_before_launch(lib):
    _, nf = ws(1, 1, 8, 16, 32, 4)
    _, nb = ws(1, 1, 8, 16, 32, 4, bwd=True)
    # B^(0): value and normaliser together, residuals only with them, aligned
    assert fwd_from_call(lib, (FAKE, None, None, None)) == INVALID
    assert fwd_from_call(lib, (None, FAKE, None, None)) == INVALID
    assert fwd_from_call(lib, (None, None, FAKE, None)) == INVALID
    assert fwd_from_call(lib, (FAKE + 4, FAKE, None, None)) == INVALID
    assert fwd_from_call(lib, (FAKE, FAKE, FAKE, None), wsb=nf - 1) == WORKSPACE
    assert fwd_from_call(lib, (None, None, None, None), wsb=nf - 1) == WORKSPACE
    # G^(N) in and G^(0) out: pairs, aligned
    assert bwd_from_call(lib, (FAKE, None), (None, None)) == INVALID
    assert bwd_from_call(lib, (None, None), (None, FAKE)) == INVALID
    assert bwd_from_call(lib, (FAKE, FAKE), (FAKE + 8, FAKE)) == INVALID
    assert bwd_from_call(lib, (FAKE, FAKE), (FAKE, FAKE), wsb=nb - 1) == WORKSPACE


def stack_ws(B, H, L, d, M, C, layers, bwd):
    n = ctypes.c_size_t(0)
    st = slim.library().slim_stack_workspace_size(B, H, L, d, M, C, layers, 0, 0, 1 if bwd else 0,
                                                   ctypes.byref(n))
    return st, n.value


def test_stack_workspace_scales_with_C_and_layers_not_L(lib):
    for bwd in (False, True):
        st, a = stack_ws(2, 2, 4096, 64, 128, 256, 3, bwd)
        assert st == OK and a > 0
        assert stack_ws(2, 2, 65536, 64, 128, 256, 3, bwd) == (OK, a)      # O(C), not O(L)
        _, b = stack_ws(2, 2, 4096, 64, 128, 512, 3, bwd)
        assert b > a
        _, c = stack_ws(2, 2, 4096, 64, 128, 256, 6, bwd)
        # the forward keeps one slice's rows (states are outputs); the backward
        # keeps every layer's slice input and output and its states
        assert c > a if bwd else c == a
    assert stack_ws(2, 2, 4096, 64, 128, 256, 0, False)[0] == INVALID
    assert stack_ws(2, 2, 4096, 64, 128, 256, 65, True)[0] == INVALID
    assert stack_ws(2, 2, 4096, 64, 128, 256, 64, True)[0] == OK


def test_stack_rejects_before_launch(lib):
    dims = (1, 1, 8, 16, 32, 4)
    _, nf = stack_ws(*dims, 2, False)
    _, nb = stack_ws(*dims, 2, True)

    def fwd(layers=2, om=FAKE, lo=(None, None), S=FAKE, wsb=nf, wsp=FAKE):
        return lib.slim_stack_fwd(FAKE, om, *dims, layers, 0, 0, FAKE, S, FAKE, lo[0], lo[1],
                                  wsp, wsb, None)

    def bwd(layers=2, om=FAKE, dom=FAKE, wsb=nb, wsp=FAKE):
        return lib.slim_stack_bwd(FAKE, om, FAKE, FAKE, FAKE, None, None, *dims, layers, 0, 0,
                                  FAKE, dom, wsp, wsb, None)

    assert fwd(layers=0) == INVALID and fwd(layers=65) == INVALID
    assert fwd(om=None) == INVALID                  # Omega needed for exp features
    assert fwd(lo=(FAKE, None)) == INVALID          # residuals both or neither
    assert fwd(S=FAKE + 4) == INVALID               # misaligned state
    assert fwd(wsb=nf - 1) == WORKSPACE
    assert fwd(wsp=FAKE + 16) == INVALID            # workspace not 256-byte aligned
    assert bwd(layers=65) == INVALID
    assert bwd(dom=None) == INVALID
    assert bwd(wsb=nb - 1) == WORKSPACE
