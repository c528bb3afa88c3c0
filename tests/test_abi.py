"""The C ABI on the host: the library loads, exports every declared symbol, sizes its
workspace from the shape, and rejects bad arguments before touching the GPU.

Nothing here launches a kernel: every call below fails validation (or is a no-op shape),
so these tests run on a machine without a GPU.
"""
import ctypes
import os
import re

import pytest

from paper_2608_11519_gb300 import build as lib_build
from paper_2608_11519_gb300 import flarepp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    lib_build.build()
    return flarepp.load()


def declared_symbols():
    syms = []
    for name in os.listdir(os.path.join(ROOT, "include")):
        if name.endswith(".h"):
            text = open(os.path.join(ROOT, "include", name)).read()
            syms += re.findall(r"FLAREPP_API\s+[\w\s\*]+?\b(flarepp_\w+)\s*\(", text)
    return sorted(set(syms))


def test_every_declared_symbol_is_exported(lib):
    syms = declared_symbols()
    assert len(syms) >= 6
    for s in syms:
        assert hasattr(lib, s), s
    assert set(flarepp.EXPORTED) <= set(syms)


def test_status_strings(lib):
    for code in range(6):
        assert flarepp.status_string(code)
    assert flarepp.status_string(99) == "unknown status"
    assert flarepp.version().count(".") == 2


def S(B=1, H=2, N=1000, M=32, D=32, dtype=flarepp.BF16):
    return flarepp.Shape(B, H, N, M, D, dtype)


def test_workspace_bytes(lib):
    ws = lambda s: lib.flarepp_route_workspace_bytes(ctypes.byref(s))
    assert ws(S()) > 0
    assert ws(S()) % 256 == 0
    # invalid or unsupported shapes need none
    assert ws(S(D=24)) == 0
    assert ws(S(M=4096)) == 0
    assert ws(S(B=-1)) == 0
    assert ws(S(dtype=7)) == 0
    assert lib.flarepp_route_workspace_bytes(None) == 0
    # degenerate shapes need none
    assert ws(S(N=0)) == 0 and ws(S(B=0)) == 0 and ws(S(M=0)) == 0
    # grows with the problem; holds at least Q and Z in float32
    small, big = ws(S(N=1000)), ws(S(N=1000, M=1024))
    assert big > small >= 2 * 1 * 2 * 32 * 32 * 4
    # a function of the shape alone
    assert ws(S(B=4, H=8, N=16384, M=128)) == ws(S(B=4, H=8, N=16384, M=128))


FAKE = 0x7F0000000000  # an aligned address that is never dereferenced


def call(lib, shape, ptrs=None, scale=0.25, ws=None, ws_bytes=None, Y=None):
    p = ptrs or {}
    base = FAKE
    vals = {}
    for i, n in enumerate(("seeds", "Kt", "Vt", "K", "V")):
        vals[n] = p.get(n, base + (i + 1) * (1 << 36))
    Yp = Y if Y is not None else base + 6 * (1 << 36)
    wsp = ws if ws is not None else base + 7 * (1 << 36)
    need = lib.flarepp_route_workspace_bytes(ctypes.byref(shape)) if shape is not None else 0
    wsb = need if ws_bytes is None else ws_bytes
    v = lambda x: None if x is None else ctypes.c_void_p(x)
    return lib.flarepp_route_fwd(None if shape is None else ctypes.byref(shape), v(vals["seeds"]),
                                 v(vals["Kt"]), v(vals["Vt"]), v(vals["K"]), v(vals["V"]),
                                 ctypes.c_float(scale), v(Yp), v(wsp), wsb, None)


def test_invalid_arguments_rejected_before_launch(lib):
    E = flarepp
    assert call(lib, None) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(dtype=3)) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(N=-5)) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(D=48)) == E.ERR_UNSUPPORTED
    assert call(lib, S(D=128)) == E.ERR_UNSUPPORTED
    assert call(lib, S(M=2049)) == E.ERR_UNSUPPORTED
    assert call(lib, S(B=1 << 20, H=1 << 20, N=1 << 20)) == E.ERR_UNSUPPORTED
    assert call(lib, S(), scale=float("nan")) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(), scale=float("inf")) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(), ptrs={"K": None}) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(), ptrs={"seeds": None}) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(), ptrs={"V": FAKE + 8}) == E.ERR_INVALID_ARGUMENT  # misaligned
    assert call(lib, S(), Y=FAKE + (1 << 36) + 64) == E.ERR_INVALID_ARGUMENT  # Y overlaps Kt...
    assert call(lib, S(), Y=FAKE + 1 * (1 << 36)) == E.ERR_INVALID_ARGUMENT
    assert call(lib, S(), ws_bytes=16) == E.ERR_WORKSPACE
    assert call(lib, S(), ws=FAKE + 7 * (1 << 36) + 128) == E.ERR_WORKSPACE  # not 256-aligned
    assert call(lib, S(), ws=0) == E.ERR_WORKSPACE
    # the kernels write the workspace while they read the inputs
    assert call(lib, S(), ws=FAKE + 4 * (1 << 36)) == E.ERR_INVALID_ARGUMENT  # workspace on K
    assert call(lib, S(), ws=FAKE + (1 << 36) - 256) == E.ERR_INVALID_ARGUMENT  # ends in seeds
    # the debug entry's Q and Z copies may not land on the workspace or on Y
    dbg = lambda q, z: lib.flarepp_route_fwd_debug(
        ctypes.byref(S()), *(ctypes.c_void_p(FAKE + (i + 1) * (1 << 36)) for i in range(5)),
        ctypes.c_float(0.25), ctypes.c_void_p(FAKE + 6 * (1 << 36)),
        ctypes.c_void_p(FAKE + 7 * (1 << 36)), lib.flarepp_route_workspace_bytes(ctypes.byref(S())),
        None, None if q is None else ctypes.c_void_p(q), None if z is None else ctypes.c_void_p(z))
    assert dbg(FAKE + 7 * (1 << 36) + 256, None) == E.ERR_INVALID_ARGUMENT
    assert dbg(None, FAKE + 6 * (1 << 36) + 64) == E.ERR_INVALID_ARGUMENT
    # FLARE: the same rules through its own entry (Q, K, V, Y, workspace)
    fl = lambda ws: lib.flarepp_flare_fwd(
        ctypes.byref(S()), *(ctypes.c_void_p(FAKE + (i + 1) * (1 << 36)) for i in range(3)),
        ctypes.c_float(0.25), ctypes.c_void_p(FAKE + 6 * (1 << 36)), ctypes.c_void_p(ws),
        lib.flarepp_route_workspace_bytes(ctypes.byref(S())), None, None)
    assert fl(FAKE + 3 * (1 << 36)) == E.ERR_INVALID_ARGUMENT  # workspace on V
    assert fl(FAKE + 6 * (1 << 36)) == E.ERR_INVALID_ARGUMENT  # workspace on Y
    # profiled entry: events required
    assert lib.flarepp_route_fwd_profiled(ctypes.byref(S()), None, None, None, None, None,
                                          ctypes.c_float(0.25), None, None, 0, None, None,
                                          6) == E.ERR_INVALID_ARGUMENT


def test_degenerate_shapes_are_noops(lib):
    # B*H = 0 and N = 0 enqueue nothing, so they succeed even without a GPU
    assert call(lib, S(B=0)) == flarepp.OK
    assert call(lib, S(H=0)) == flarepp.OK
    assert call(lib, S(N=0), ptrs={k: None for k in ("Kt", "Vt", "K", "V")}) == flarepp.OK


def test_python_binding_rejects_bad_tensors(lib):
    import torch
    x = torch.zeros(1, 2, 8, 32, dtype=torch.bfloat16)
    s = torch.zeros(2, 4, 32, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        flarepp.route_fwd(s, x, x, x, x)  # host tensors
    with pytest.raises(TypeError):
        flarepp.route_fwd(s, x, x, x.float(), x)
    with pytest.raises(ValueError):
        flarepp.route_fwd(s[:1], x, x, x, x)
    with pytest.raises(ValueError):
        flarepp.route_fwd(s, x.transpose(2, 3), x, x, x)
    # caller-supplied outputs are checked before the device is looked at: a short Y would
    # be written past its end
    short = torch.zeros(1, 2, 4, 32, dtype=torch.bfloat16)
    for f in (flarepp.route_fwd, flarepp.route_fwd_train, flarepp.route_fwd_noalloc):
        with pytest.raises(ValueError, match="Y must"):
            f(s, x, x, x, x, Y=short)
    with pytest.raises(ValueError, match="Y must"):
        flarepp.route_fwd(s, x, x, x, x, Y=x.float())
    with pytest.raises(ValueError, match="Y must"):
        flarepp.flare_fwd(s, x, x, Y=x.transpose(2, 3))
    with pytest.raises(ValueError, match="grads must"):
        flarepp.route_bwd(s, x, x, x, x, x, x, None, grads=(s, x, x, x))
    with pytest.raises(ValueError, match="dV must"):
        flarepp.route_bwd(s, x, x, x, x, x, x, None, grads=(s, x, x, x, short))
    X = torch.zeros(1, 8, 64, dtype=torch.bfloat16)
    W = torch.zeros(4 * 64, 64, dtype=torch.bfloat16)
    Wo = torch.zeros(64, 64, dtype=torch.bfloat16)
    sd = torch.zeros(2, 4, 32, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="O must"):
        flarepp.mixer_fwd(X, W, Wo, sd, O=X[:, :4])
    with pytest.raises(ValueError, match="O must"):
        flarepp.mixer_fwd_train(X, W, Wo, sd, O=X.float())
    with pytest.raises(ValueError, match="dW_in must"):
        flarepp.mixer_bwd(X, W, Wo, sd, None, X, grads=(X, W[:64], Wo, sd))
    with pytest.raises(ValueError, match="expected X"):
        flarepp.mixer_fwd(X[0], W, Wo, sd)
    # well-formed host tensors still reach the device check
    for f, a in ((flarepp.mixer_fwd, (X, W, Wo, sd)), (flarepp.route_fwd, (s, x, x, x, x))):
        with pytest.raises(ValueError, match="takes device tensors"):
            f(*a)


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(RuntimeError):
        flarepp.load(str(tmp_path / "libflarepp.so"))


def test_host_entry_sizes_and_rejects_before_any_cuda_call(lib):
    E = flarepp
    hb = lambda s: lib.flarepp_route_host_buffer_bytes(ctypes.byref(s))
    # the device buffer holds a group's workspace plus device copies of the inputs and Y
    s = S(B=1, H=8, N=5000, M=128, D=32)
    tok = 1 * 8 * 5000 * 32 * 2
    assert hb(s) >= 5 * tok and hb(s) % 256 == 0
    assert hb(S(D=48)) == 0 and hb(S(N=0)) == 0 and hb(S(B=0)) == 0

    def host_call(shape, Y=FAKE + 6 * (1 << 36), buf=FAKE + 7 * (1 << 36), nbytes=None,
                  scale=0.25):
        ptrs = [ctypes.c_void_p(FAKE + (i + 1) * (1 << 36)) for i in range(5)]
        nb = hb(shape) if nbytes is None else nbytes
        return lib.flarepp_route_fwd_host(ctypes.byref(shape), *ptrs, ctypes.c_float(scale),
                                          ctypes.c_void_p(Y) if Y else None,
                                          ctypes.c_void_p(buf) if buf else None, nb, None)

    assert host_call(S(D=48)) == E.ERR_UNSUPPORTED
    assert host_call(S(), scale=float("nan")) == E.ERR_INVALID_ARGUMENT
    assert host_call(S(), Y=0) == E.ERR_INVALID_ARGUMENT
    assert host_call(S(), Y=FAKE + (1 << 36) + 64) == E.ERR_INVALID_ARGUMENT  # Y overlaps Kt
    assert host_call(S(), buf=0) == E.ERR_WORKSPACE
    assert host_call(S(), nbytes=1024) == E.ERR_WORKSPACE
    assert host_call(S(), buf=FAKE + 7 * (1 << 36) + 128) == E.ERR_WORKSPACE  # not aligned
    assert host_call(S(N=0)) == E.OK  # empty Y: nothing to do

    # FLARE on host buffers: the same checks through its own entry (Q, K, V, then Y)
    def flare_host_call(shape, Y=FAKE + 6 * (1 << 36), buf=FAKE + 7 * (1 << 36), nbytes=None,
                        scale=0.25):
        ptrs = [ctypes.c_void_p(FAKE + (i + 1) * (1 << 36)) for i in range(3)]
        nb = hb(shape) if nbytes is None else nbytes
        return lib.flarepp_flare_fwd_host(ctypes.byref(shape), *ptrs, ctypes.c_float(scale),
                                          ctypes.c_void_p(Y) if Y else None,
                                          ctypes.c_void_p(buf) if buf else None, nb, None)

    assert flare_host_call(S(D=48)) == E.ERR_UNSUPPORTED
    assert flare_host_call(S(), scale=float("inf")) == E.ERR_INVALID_ARGUMENT
    assert flare_host_call(S(), Y=0) == E.ERR_INVALID_ARGUMENT
    assert flare_host_call(S(), Y=FAKE + 2 * (1 << 36) + 64) == E.ERR_INVALID_ARGUMENT  # Y on K
    assert flare_host_call(S(), buf=0) == E.ERR_WORKSPACE
    assert flare_host_call(S(), nbytes=1024) == E.ERR_WORKSPACE
    assert flare_host_call(S(N=0)) == E.OK


def test_backward_entry_sizes_and_rejects_before_any_cuda_call(lib):
    E = flarepp
    sb = lambda s: lib.flarepp_route_saved_bytes(ctypes.byref(s))
    wb = lambda s: lib.flarepp_route_bwd_workspace_bytes(ctypes.byref(s))
    s = S(B=2, H=3, N=1000, M=40, D=32)
    # saved: Q, Z float32 [B,H,M,D], L1, L2 [B,H,M], L3 [B,H,N]
    assert sb(s) >= (2 * 6 * 40 * 32 + 2 * 6 * 40 + 6 * 1000) * 4
    assert wb(s) > 0 and wb(s) % 256 == 0
    assert sb(S(N=0)) == 0 and sb(S(D=48)) == 0 and wb(S(D=48)) == 0

    base = [FAKE + (i + 1) * (1 << 36) for i in range(14)]

    def bwd(shape, ptrs=None, saved_bytes=None, ws_bytes=None, scale=0.25):
        p = list(base) if ptrs is None else ptrs
        v = lambda x: None if x is None else ctypes.c_void_p(x)
        # seeds Kt Vt K V Y dY saved | dseeds dKt dVt dK dV | workspace
        return lib.flarepp_route_bwd(
            ctypes.byref(shape), *(v(x) for x in p[:5]), ctypes.c_float(scale), v(p[5]),
            v(p[6]), v(p[7]), sb(shape) if saved_bytes is None else saved_bytes,
            *(v(x) for x in p[8:13]), v(p[13]), wb(shape) if ws_bytes is None else ws_bytes,
            None)

    assert bwd(S(D=48)) == E.ERR_UNSUPPORTED
    assert bwd(S(), scale=float("nan")) == E.ERR_INVALID_ARGUMENT
    for i in range(13):  # every pointer is required
        p = list(base)
        p[i] = None
        assert bwd(S(), p) == E.ERR_INVALID_ARGUMENT, i
    p = list(base)
    p[9] = base[1] + 64  # dKt overlaps Kt
    assert bwd(S(), p) == E.ERR_INVALID_ARGUMENT
    p = list(base)
    p[11] = base[10] + 16  # dK overlaps dVt
    assert bwd(S(), p) == E.ERR_INVALID_ARGUMENT
    p = list(base)
    p[12] = base[8] + 8  # misaligned dV
    assert bwd(S(), p) == E.ERR_INVALID_ARGUMENT
    assert bwd(S(), saved_bytes=16) == E.ERR_INVALID_ARGUMENT
    assert bwd(S(), ws_bytes=16) == E.ERR_WORKSPACE
    p = list(base)
    p[13] = None
    assert bwd(S(), p) == E.ERR_WORKSPACE
    for i in (5, 6, 7):  # the workspace on Y, dY or saved
        p = list(base)
        p[13] = base[i]
        assert bwd(S(), p) == E.ERR_INVALID_ARGUMENT, i
    # the training forward checks its saved buffer
    v = lambda x: ctypes.c_void_p(x)
    fw = lambda saved, nbytes: lib.flarepp_route_fwd_train(
        ctypes.byref(S()), *(v(x) for x in base[:5]), ctypes.c_float(0.25), v(base[5]),
        None if saved is None else v(saved), nbytes, v(base[13]),
        lib.flarepp_route_workspace_bytes(ctypes.byref(S())), None)
    assert fw(None, sb(S())) == E.ERR_INVALID_ARGUMENT
    assert fw(base[7], 16) == E.ERR_INVALID_ARGUMENT
    assert fw(base[1] + 32, sb(S())) == E.ERR_INVALID_ARGUMENT  # overlaps Kt


def test_mixer_entry_sizes_and_rejects(lib):
    E = flarepp
    wb = lambda s, p: lib.flarepp_mixer_workspace_bytes(ctypes.byref(s), p)
    s = S(B=1, H=8, N=4096, M=64, D=32)
    tok = 8 * 4096 * 32 * 2
    assert wb(s, 4) >= 5 * tok and wb(s, 2) >= 3 * tok and wb(s, 4) > wb(s, 2)
    assert wb(s, 3) == 0 and wb(S(dtype=flarepp.F32), 4) == 0 and wb(S(N=0), 4) == 0
    v = lambda x: ctypes.c_void_p(x)
    ptr = [FAKE + (i + 1) * (1 << 36) for i in range(6)]

    def call(shape, n_proj=4, scale=0.25, ptrs=None):
        p = ptr if ptrs is None else ptrs
        return lib.flarepp_mixer_fwd(ctypes.byref(shape), n_proj, *(v(x) if x else None
                                                                    for x in p[:4]),
                                     ctypes.c_float(scale), v(p[4]) if p[4] else None,
                                     v(p[5]) if p[5] else None, wb(shape, n_proj), None)

    assert call(S(dtype=flarepp.F32)) == E.ERR_UNSUPPORTED
    assert call(S(), n_proj=3) == E.ERR_INVALID_ARGUMENT
    assert call(S(), scale=float("inf")) == E.ERR_INVALID_ARGUMENT
    for i in range(5):
        p = list(ptr)
        p[i] = None
        assert call(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT, i
    p = list(ptr)
    p[4] = ptr[0] + 64  # O overlaps X
    assert call(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT
    p = list(ptr)
    p[5] = None
    assert call(S(), ptrs=p) == E.ERR_WORKSPACE
    for i in range(4):  # the workspace on X, W_in, Wo or seeds
        p = list(ptr)
        p[5] = ptr[i]
        assert call(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT, i


def test_mixer_training_entries_reject(lib):
    E = flarepp
    s = S(B=1, H=8, N=4096, M=64, D=32)
    sb = lambda sh, p: lib.flarepp_mixer_saved_bytes(ctypes.byref(sh), p)
    wb = lambda sh, p: lib.flarepp_mixer_bwd_workspace_bytes(ctypes.byref(sh), p)
    # the saved state holds Y and the projections (two more for n_proj = 4)
    tok = 8 * 4096 * 32 * 2
    assert sb(s, 4) - sb(s, 2) == 2 * tok and sb(s, 2) > 3 * tok
    assert wb(s, 4) == wb(s, 2) > 0
    assert sb(s, 3) == 0 and wb(S(dtype=flarepp.F32), 4) == 0 and wb(S(N=0), 4) == 0
    v = lambda x: ctypes.c_void_p(x) if x else None
    base = [FAKE + (i + 1) * (1 << 36) for i in range(11)]

    def bwd(shape, n_proj=4, ptrs=None, scale=0.25, saved_bytes=None):
        p = base if ptrs is None else ptrs
        # X W_in Wo seeds | saved | dO | dX dW_in dWo dseeds | workspace
        return lib.flarepp_mixer_bwd(
            ctypes.byref(shape), n_proj, *(v(x) for x in p[:4]), ctypes.c_float(scale), v(p[4]),
            sb(shape, n_proj) if saved_bytes is None else saved_bytes, v(p[5]),
            *(v(x) for x in p[6:10]), v(p[10]), wb(shape, n_proj), None)

    assert bwd(S(dtype=flarepp.F32)) == E.ERR_UNSUPPORTED
    assert bwd(S(), n_proj=3) == E.ERR_INVALID_ARGUMENT
    assert bwd(S(), scale=float("nan")) == E.ERR_INVALID_ARGUMENT
    for i in (0, 1, 2, 3, 5, 6, 7, 8, 9):
        p = list(base)
        p[i] = None
        assert bwd(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT, i
    p = list(base)
    p[6] = base[0] + 32  # dX overlaps X
    assert bwd(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT
    assert bwd(S(), saved_bytes=16) == E.ERR_INVALID_ARGUMENT
    p = list(base)
    p[10] = None
    assert bwd(S(), ptrs=p) == E.ERR_WORKSPACE
    for i in (0, 4, 5, 6, 9):  # the workspace on X, saved, dO, dX or dseeds
        p = list(base)
        p[10] = base[i]
        assert bwd(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT, i
    for i in (6, 9):  # dX or dseeds on saved
        p = list(base)
        p[i] = base[4] + 64
        assert bwd(S(), ptrs=p) == E.ERR_INVALID_ARGUMENT, i
