"""The C ABI library builds, loads and exports every declared entry point;
host-side validation rejects bad arguments before touching any GPU."""
import ctypes
import os
import re

import pytest

from paper_2608_23794_gb300 import build as moce_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moce.h")


@pytest.fixture(scope="module")
def lib():
    path = moce_build.build()
    return ctypes.CDLL(path)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(moce_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("moce_pack_supports", "moce_pool", "moce_gate", "moce_forward",
                     "moce_workspace_bytes", "moce_status_string", "moce_check_device_error"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_carries_every_entry_point_by_name(lib):
    """The Python binding has a function of the same name for every declared entry point; the
    ones that need no device answer like the library."""
    from paper_2608_23794_gb300 import moce
    for name in declared_functions():
        assert callable(getattr(moce, name, None)), name
    assert moce.moce_status_string(2) == "MOCE_ERR_BAD_SUPPORT"
    lib.moce_pack_workspace_bytes.argtypes = [ctypes.c_int] * 3
    lib.moce_pack_workspace_bytes.restype = ctypes.c_size_t
    assert moce.moce_pack_workspace_bytes(64, 16, 4) == lib.moce_pack_workspace_bytes(64, 16, 4) > 0
    assert moce.moce_pack_workspace_bytes(0, 16, 4) == 0
    assert moce.moce_train_workspace_bytes(256, 64) > 0
    total = moce.moce_workspace_bytes(2, 8, 8, 64, 16, 4)
    z_off, tau_off = moce.moce_workspace_offsets(2, 8, 8, 64, 16, 4)
    assert z_off % 4 == 0 and tau_off % 4 == 0
    assert z_off + 4 * 2 * 64 <= total and tau_off + 4 * 2 * 16 <= total
    assert z_off + 4 * 2 * 64 <= tau_off or tau_off + 4 * 2 * 16 <= z_off
    ws = moce.Workspace(2, 8, 8, 64, 16, 4, device="cpu")  # host buffer: offsets only
    assert (ws.z_offset, ws.tau_offset, ws.nbytes) == (z_off, tau_off, total)
    with pytest.raises(ValueError):  # the library is never handed a host buffer
        moce.moce_workspace_init(ws)


def test_status_strings(lib):
    lib.moce_status_string.restype = ctypes.c_char_p
    lib.moce_status_string.argtypes = [ctypes.c_int]
    assert lib.moce_status_string(0) == b"MOCE_OK"
    assert lib.moce_status_string(2) == b"MOCE_ERR_BAD_SUPPORT"
    assert lib.moce_status_string(99) == b"MOCE_ERR_UNKNOWN"


def test_workspace_bytes(lib):
    f = lib.moce_workspace_bytes
    f.restype = ctypes.c_size_t
    f.argtypes = [ctypes.c_int] * 6
    n = f(64, 56, 56, 256, 64, 16)
    # z + tau + mixing weights + pooling partials at least
    assert n >= 64 * 256 * 4 + 64 * 64 * 4 + 64 * 64 * 16 * 4
    assert n % 256 == 0
    assert f(64, 56, 56, 256, 64, 0) == 0          # k < 1
    assert f(64, 56, 56, 256, 64, 257) == 0        # k > C_in
    assert f(1, 1, 1, 70000, 4, 2) == 0            # C_in beyond 16-bit indices
    pf = lib.moce_pack_workspace_bytes
    pf.restype = ctypes.c_size_t
    pf.argtypes = [ctypes.c_int] * 3
    assert pf(256, 64, 16) >= 4 * (2 + 256 // 32)


def test_forward_rejects_bad_arguments_on_host(lib):
    f = lib.moce_forward
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    f.argtypes = [P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F, P, P, ctypes.c_size_t, P]
    f.restype = I
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: validation fails first
    good = dict(x=fake, N=2, H=4, W=4, C=64, R=8, k=4, dt=1, lay=0, tmin=0.2, tmax=6.0)

    def call(**kw):
        a = {**good, **kw}
        return f(a["x"], a["N"], a["H"], a["W"], a["C"], a["R"], a["k"], a["dt"], a["lay"], fake,
                 fake, fake, 3, fake, fake, fake, fake, a["tmin"], a["tmax"], fake, fake, 0, None)

    assert call(k=0) == 1
    assert call(k=65) == 1
    assert call(R=0) == 1
    assert call(dt=7) == 1
    assert call(lay=3) == 1
    assert call(tmin=0.0) == 1
    assert call(tmin=7.0) == 1
    assert call(tmax=float("inf")) == 1
    assert call(x=None) == 1
    assert call() == 1  # workspace of 0 bytes is too small
    assert call(N=0) == 0  # empty batch: nothing to do


def test_forward_path_selection_on_host(lib):
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    f = lib.moce_forward_path
    f.argtypes = [P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F, P, P, ctypes.c_size_t,
                  I, P]
    f.restype = I
    n = lib.moce_forward_path_launches
    n.argtypes = [P, I, I, I, I, I, I, I, I, I]
    n.restype = I
    name = lib.moce_forward_path_kernel
    name.argtypes = n.argtypes
    name.restype = ctypes.c_char_p
    fake = ctypes.c_void_p(0x1000)  # 256-byte aligned, never dereferenced

    def call(dt, path, ws_bytes=1 << 40):
        return f(fake, 2, 8, 8, 64, 16, 4, dt, 0, fake, fake, fake, 3, fake, fake, fake, fake,
                 0.2, 6.0, fake, fake, ws_bytes, path, None)

    assert call(1, 7) == 1             # not a path
    for retired in (1, 2, 3, 5):       # values of kernels this library no longer has
        assert call(1, retired) == 1
        assert n(fake, 2, 8, 8, 64, 16, 4, 1, 0, retired) == 0
    assert call(1, -1) == 1
    # without a GPU the stream kernel cannot be planned (no SM count, no
    # tensor-map encoder): unsupported, nothing enqueued; AUTO takes the steps
    assert call(1, 6) == 3
    assert n(fake, 2, 8, 8, 64, 16, 4, 1, 0, 6) == 0
    assert name(fake, 2, 8, 8, 64, 16, 4, 1, 0, 6) is None
    assert n(fake, 2, 8, 8, 64, 16, 4, 1, 0, 0) == 3   # pool (one span per example), gate, mix
    assert name(fake, 2, 8, 8, 64, 16, 4, 1, 0, 0) == b"pool+gate+mix"
    assert n(fake, 2, 8, 8, 64, 16, 4, 1, 0, 4) == 3
    # two examples of 56 x 56 positions: the pool splits each into spans whose tile sums a
    # second kernel adds
    assert n(fake, 2, 56, 56, 256, 16, 4, 1, 0, 4) == 4
    # 160 examples of 7 x 7 x 1024: enough CTAs with one span per example
    assert n(fake, 160, 7, 7, 1024, 16, 4, 1, 0, 4) == 3
    # fp32 has no stream kernel either; the steps run any dtype, layout and alignment
    assert call(0, 6) == 3
    odd = ctypes.c_void_p(0x1002)
    assert n(odd, 2, 8, 8, 64, 16, 4, 1, 0, 6) == 0
    assert n(odd, 2, 8, 8, 64, 16, 4, 1, 0, 4) == 3
    assert n(fake, 2, 8, 8, 64, 16, 4, 1, 1, 6) == 0
    assert n(fake, 2, 8, 8, 64, 16, 4, 1, 1, 0) == 3   # NCHW: pool, gate, mix


def test_backward_rejects_bad_arguments_on_host(lib):
    P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    wb = lib.moce_backward_workspace_bytes
    wb.argtypes, wb.restype = [I] * 6, S
    f = lib.moce_backward
    f.argtypes = [P, P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F,
                  P, P, P, P, P, P, P, S, P]
    f.restype = I
    assert wb(2, 4, 4, 64, 8, 4) > 0
    assert wb(2, 4, 4, 64, 8, 0) == 0            # k < 1
    assert wb(2, 4, 4, 6000, 8, 4) == 0          # staged da tile does not fit
    assert wb(2, 4, 4, 64, 3500, 4) == 0         # staged dy tile of dx does not fit
    fake = ctypes.c_void_p(0x1000)
    good = dict(N=2, H=4, W=4, C=64, R=8, k=4, dt=1, lay=0, tmin=0.2, tmax=6.0, nU=3, dx=fake,
                dW1=fake, ws=fake, wsb=1 << 40)

    def call(**kw):
        a = {**good, **kw}
        return f(fake, fake, a["N"], a["H"], a["W"], a["C"], a["R"], a["k"], a["dt"], a["lay"],
                 fake, fake, fake, a["nU"], fake, fake, fake, fake, a["tmin"], a["tmax"], a["dx"],
                 fake, a["dW1"], fake, fake, fake, a["ws"], a["wsb"], None)

    assert call(k=0) == 1
    assert call(k=65) == 1
    assert call(dt=5) == 1
    assert call(lay=2) == 1
    assert call(tmin=-1.0) == 1
    assert call(nU=-1) == 1
    assert call(nU=65) == 1
    assert call(dW1=None) == 1
    assert call(dx=None) == 1
    assert call(ws=None) == 1
    assert call(wsb=16) == 1                      # workspace too small
    assert call(ws=ctypes.c_void_p(0x1010)) == 1  # not 256-byte aligned
    assert call(C=6000, nU=0) == 3                # valid, no kernel for it


def test_dynamic_rejects_bad_arguments_on_host(lib):
    P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    wb = lib.moce_dynamic_workspace_bytes
    wb.argtypes, wb.restype = [I] * 7, S
    assert wb(2, 4, 4, 64, 8, 4, 16) > 0
    assert wb(2, 4, 4, 64, 8, 4, 0) == 0          # d < 1
    assert wb(2, 4, 4, 60000, 8, 4, 16) == 0      # C_in beyond the shared-memory TopK
    # the routing buffers do not depend on H, W: a larger H W only adds the forward part
    assert wb(2, 64, 64, 64, 8, 4, 16) > wb(2, 4, 4, 64, 8, 4, 16)
    f = lib.moce_forward_dynamic
    f.argtypes = [P, I, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, P, P, F, F, P, P, P, P, P, S, P]
    f.restype = I
    fake = ctypes.c_void_p(0x1000)
    good = dict(N=2, C=64, R=8, k=4, d=16, dt=1, lay=0, tmin=0.2, tmax=6.0, ws=fake, wsb=1 << 40)

    def call(**kw):
        a = {**good, **kw}
        return f(fake, a["N"], 4, 4, a["C"], a["R"], a["k"], a["d"], a["dt"], a["lay"], fake, fake,
                 fake, fake, fake, fake, fake, fake, fake, a["tmin"], a["tmax"], fake, None, None,
                 None, a["ws"], a["wsb"], None)

    assert call(d=0) == 1
    assert call(k=65) == 1
    assert call(dt=3) == 1
    assert call(tmin=0.0) == 1
    assert call(ws=None) == 1
    assert call(wsb=64) == 1
    assert call(ws=ctypes.c_void_p(0x1080)) == 1     # not 256-byte aligned
    assert call(C=60000, k=4) == 3                    # valid, TopK row does not fit
    assert call(N=0) == 0
    m = lib.moce_mix
    m.argtypes = [P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, S, P]
    m.restype = I
    assert m(fake, 2, 4, 4, 64, 8, 4, 1, 0, fake, fake, fake, 65, None, fake, fake, 1 << 40,
             None) == 1                               # |U| > C_in
    assert m(fake, 2, 4, 4, 64, 8, 4, 1, 0, fake, fake, None, 0, fake, fake, fake, 1 << 40,
             None) == 1                               # per-example U without its rows


def test_pack_rejects_bad_arguments_on_host(lib):
    f = lib.moce_pack_supports
    P, I = ctypes.c_void_p, ctypes.c_int
    f.argtypes = [I, I, I, P, P, P, P, P, P, P, ctypes.c_size_t, P]
    f.restype = I
    fake = ctypes.c_void_p(0x1000)
    n = ctypes.c_int32(0)
    assert f(64, 8, 0, fake, fake, fake, fake, fake, ctypes.byref(n), fake, 4096, None) == 1
    assert f(64, 8, 4, None, fake, fake, fake, fake, ctypes.byref(n), fake, 4096, None) == 1
    assert f(64, 8, 4, fake, fake, fake, fake, fake, ctypes.byref(n), fake, 4, None) == 1


def test_binding_refuses_cpu_tensors():
    torch = pytest.importorskip("torch")
    from paper_2608_23794_gb300 import moce
    x = torch.zeros((1, 2, 2, 8), dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        moce._ptr(x)
