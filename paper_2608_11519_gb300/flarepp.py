"""Python binding of libflarepp (ctypes): argument marshalling only.

Every step of the routing chain runs in the library's CUDA kernels. PyTorch provides the
device memory and the stream. There is no fallback: if the library is not built, every
call raises.

    from paper_2608_11519_gb300 import flarepp
    Y = flarepp.route_fwd(seeds, Kt, Vt, K, V)              # device tensors
    Y, Q, Z = flarepp.route_fwd_debug(seeds, Kt, Vt, K, V)  # plus the intermediates
    Y = flarepp.route_fwd_host(seeds, Kt, Vt, K, V)         # host tensors in, host Y out
"""
import ctypes
import functools
import inspect
import math
import os

import torch

from . import build as _build

F32, BF16 = 0, 1
OK, ERR_INVALID_ARGUMENT, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT = range(6)
_DTYPES = {torch.float32: F32, torch.bfloat16: BF16}

EXPORTED = ("flarepp_route_workspace_bytes", "flarepp_route_fwd", "flarepp_route_fwd_debug",
            "flarepp_route_fwd_profiled", "flarepp_route_fwd_noalloc",
            "flarepp_flare_fwd", "flarepp_route_host_buffer_bytes", "flarepp_route_fwd_host",
            "flarepp_flare_fwd_host",
            "flarepp_mixer_workspace_bytes", "flarepp_mixer_fwd", "flarepp_mixer_fwd_profiled",
            "flarepp_mixer_saved_bytes", "flarepp_mixer_fwd_train",
            "flarepp_mixer_bwd_workspace_bytes", "flarepp_mixer_bwd",
            "flarepp_route_saved_bytes", "flarepp_route_fwd_train",
            "flarepp_route_bwd_workspace_bytes", "flarepp_route_bwd",
            "flarepp_route_device_status", "flarepp_status_string", "flarepp_version")
N_STAGE_EVENTS = 6
STAGES = ("encode1", "combine1", "encode2", "combine2", "decode")


class Shape(ctypes.Structure):
    """Mirror of ``flarepp_shape`` in include/flarepp.h."""
    _fields_ = [("B", ctypes.c_int64), ("H", ctypes.c_int64), ("N", ctypes.c_int64),
                ("M", ctypes.c_int64), ("D", ctypes.c_int64), ("dtype", ctypes.c_int32)]


class FlareppError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: status {status} ({status_string(status)})")
        self.status = status


_LIB = None


def lib_path() -> str:
    return _build.lib_path()


def load(path: str = None):
    """Load libflarepp.so (built by ``build.build()``); raises if it is missing."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    path = path or lib_path()
    if not os.path.exists(path):
        raise RuntimeError(f"libflarepp is not built ({path} missing); run "
                           "`python -c 'import __graft_entry__ as g; g.build()'` first")
    lib = ctypes.CDLL(path)
    vp, sz = ctypes.c_void_p, ctypes.c_size_t
    sp = ctypes.POINTER(Shape)
    lib.flarepp_route_workspace_bytes.restype = sz
    lib.flarepp_route_workspace_bytes.argtypes = [sp]
    lib.flarepp_route_fwd.restype = ctypes.c_int
    lib.flarepp_route_fwd.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, sz, vp]
    lib.flarepp_route_fwd_debug.restype = ctypes.c_int
    lib.flarepp_route_fwd_debug.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, sz,
                                            vp, vp, vp]
    lib.flarepp_route_fwd_profiled.restype = ctypes.c_int
    lib.flarepp_route_fwd_profiled.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, sz,
                                               vp, ctypes.POINTER(ctypes.c_void_p), ctypes.c_int]
    lib.flarepp_test_wait_fault.restype = None
    lib.flarepp_test_wait_fault.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_uint64]
    lib.flarepp_route_fwd_noalloc.restype = ctypes.c_int
    lib.flarepp_route_fwd_noalloc.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp]
    lib.flarepp_flare_fwd.restype = ctypes.c_int
    lib.flarepp_flare_fwd.argtypes = [sp, vp, vp, vp, ctypes.c_float, vp, vp, sz, vp, vp]
    lib.flarepp_route_host_buffer_bytes.restype = sz
    lib.flarepp_route_host_buffer_bytes.argtypes = [sp]
    lib.flarepp_route_fwd_host.restype = ctypes.c_int
    lib.flarepp_route_fwd_host.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, sz, vp]
    lib.flarepp_flare_fwd_host.restype = ctypes.c_int
    lib.flarepp_flare_fwd_host.argtypes = [sp, vp, vp, vp, ctypes.c_float, vp, vp, sz, vp]
    lib.flarepp_mixer_workspace_bytes.restype = sz
    lib.flarepp_mixer_workspace_bytes.argtypes = [sp, ctypes.c_int]
    lib.flarepp_mixer_fwd.restype = ctypes.c_int
    lib.flarepp_mixer_fwd.argtypes = [sp, ctypes.c_int, vp, vp, vp, vp, ctypes.c_float, vp, vp,
                                      sz, vp]
    lib.flarepp_mixer_fwd_profiled.restype = ctypes.c_int
    lib.flarepp_mixer_fwd_profiled.argtypes = [sp, ctypes.c_int, vp, vp, vp, vp, ctypes.c_float,
                                               vp, vp, sz, vp, ctypes.POINTER(ctypes.c_void_p),
                                               ctypes.c_int]
    lib.flarepp_mixer_saved_bytes.restype = sz
    lib.flarepp_mixer_saved_bytes.argtypes = [sp, ctypes.c_int]
    lib.flarepp_mixer_fwd_train.restype = ctypes.c_int
    lib.flarepp_mixer_fwd_train.argtypes = [sp, ctypes.c_int, vp, vp, vp, vp, ctypes.c_float, vp,
                                            vp, sz, vp, sz, vp]
    lib.flarepp_mixer_bwd_workspace_bytes.restype = sz
    lib.flarepp_mixer_bwd_workspace_bytes.argtypes = [sp, ctypes.c_int]
    lib.flarepp_mixer_bwd.restype = ctypes.c_int
    lib.flarepp_mixer_bwd.argtypes = [sp, ctypes.c_int, vp, vp, vp, vp, ctypes.c_float, vp, sz,
                                      vp, vp, vp, vp, vp, vp, sz, vp]
    lib.flarepp_route_saved_bytes.restype = sz
    lib.flarepp_route_saved_bytes.argtypes = [sp]
    lib.flarepp_route_fwd_train.restype = ctypes.c_int
    lib.flarepp_route_fwd_train.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, sz,
                                            vp, sz, vp]
    lib.flarepp_route_bwd_workspace_bytes.restype = sz
    lib.flarepp_route_bwd_workspace_bytes.argtypes = [sp]
    lib.flarepp_route_bwd.restype = ctypes.c_int
    lib.flarepp_route_bwd.argtypes = [sp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, vp, sz,
                                      vp, vp, vp, vp, vp, vp, sz, vp]
    lib.flarepp_route_device_status.restype = ctypes.c_int
    lib.flarepp_route_device_status.argtypes = [sp, vp, vp, ctypes.POINTER(ctypes.c_int32)]
    lib.flarepp_status_string.restype = ctypes.c_char_p
    lib.flarepp_status_string.argtypes = [ctypes.c_int]
    lib.flarepp_version.restype = ctypes.c_char_p
    if path == lib_path():
        _LIB = lib
    return lib


def status_string(status: int) -> str:
    return load().flarepp_status_string(int(status)).decode()


def version() -> str:
    return load().flarepp_version().decode()


def make_shape(B, H, N, M, D, dtype) -> Shape:
    if isinstance(dtype, torch.dtype):
        dtype = _DTYPES[dtype]
    return Shape(int(B), int(H), int(N), int(M), int(D), int(dtype))


def workspace_bytes(B, H, N, M, D, dtype) -> int:
    return int(load().flarepp_route_workspace_bytes(ctypes.byref(make_shape(B, H, N, M, D, dtype))))


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _shape_of(seeds, Kt, Vt, K, V) -> Shape:
    for t in (seeds, Kt, Vt, K, V):
        if not isinstance(t, torch.Tensor):
            raise TypeError("inputs must be torch tensors")
        if not t.is_contiguous():
            raise ValueError("inputs must be contiguous (D innermost)")
        if t.dtype != K.dtype:
            raise TypeError("all inputs must share one dtype")
    if K.dtype not in _DTYPES:
        raise TypeError(f"unsupported dtype {K.dtype}; use float32 or bfloat16")
    if K.dim() != 4 or seeds.dim() != 3:
        raise ValueError("expected seeds [H,M,D] and Kt, Vt, K, V [B,H,N,D]")
    B, H, N, D = K.shape
    M = seeds.shape[1]
    if tuple(seeds.shape) != (H, M, D):
        raise ValueError(f"seeds shape {tuple(seeds.shape)} != {(H, M, D)}")
    for t in (Kt, Vt, V):
        if tuple(t.shape) != (B, H, N, D):
            raise ValueError(f"input shape {tuple(t.shape)} != {(B, H, N, D)}")
    return make_shape(B, H, N, M, D, K.dtype)


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


def _check_out(t, like, name):
    """A caller-supplied output: a contiguous tensor of ``like``'s shape and dtype (the kernels
    write every element of it, so a smaller buffer would be written past its end)."""
    if not isinstance(t, torch.Tensor) or tuple(t.shape) != tuple(like.shape) or \
            t.dtype != like.dtype or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous {like.dtype} tensor of shape "
                         f"{tuple(like.shape)}")
    return t


def _check_device(what, device, **tensors):
    """Every tensor a device-side call touches sits on ``device``, a CUDA device: the library
    takes raw pointers and cannot tell a host address, or another GPU's, from its own."""
    if device.type != "cuda":
        raise ValueError(f"{what} takes device tensors (the *_host entries take host tensors)")
    for name, t in tensors.items():
        if isinstance(t, torch.Tensor) and t.device != device:
            raise ValueError(f"{what}: {name} is on {t.device}, expected {device}")


def _on_device(arg):
    """Run the wrapped entry with the CUDA device of argument ``arg`` current. The library
    works on the current device (the no-allocation entry looks its scratch array up there,
    and launches go to the current device's context), so a call on tensors of another GPU
    must make that GPU current first. ``arg`` names a device tensor, or the ``device``
    argument of a host entry."""
    def wrap(fn):
        sig = inspect.signature(fn)

        @functools.wraps(fn)
        def call(*a, **kw):
            v = sig.bind_partial(*a, **kw).arguments.get(arg)
            if v is None and arg in sig.parameters:
                v = sig.parameters[arg].default
            dev = v.device if isinstance(v, torch.Tensor) else (
                torch.device(v) if isinstance(v, (str, torch.device)) else None)
            if dev is None or dev.type != "cuda" or dev.index is None:
                return fn(*a, **kw)
            with torch.cuda.device(dev):
                return fn(*a, **kw)
        return call
    return wrap


class Workspace:
    """A reusable device workspace, grown on demand (one per stream at a time)."""

    def __init__(self, device=None):
        self.device = device
        self.buf = None

    def get(self, nbytes: int, device):
        if nbytes == 0:
            return None
        if self.buf is None or self.buf.numel() < nbytes or self.buf.device != device:
            self.buf = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
        # the library wants 256-byte alignment; torch allocations are at least that aligned
        if self.buf.data_ptr() % 256 != 0:
            raise RuntimeError("workspace allocation is not 256-byte aligned")
        return self.buf


def _call(debug, seeds, Kt, Vt, K, V, scale, Y, workspace, stream, Q_out, Z_out, events=None):
    lib = load()
    shape = _shape_of(seeds, Kt, Vt, K, V)
    if Y is not None:
        _check_out(Y, K, "Y")
    _check_device("route_fwd", K.device, seeds=seeds, Kt=Kt, Vt=Vt, V=V, Y=Y, Q_out=Q_out,
                  Z_out=Z_out, workspace=workspace)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y is None:
        Y = torch.empty_like(K)
    nbytes = int(lib.flarepp_route_workspace_bytes(ctypes.byref(shape)))
    if isinstance(workspace, Workspace):
        ws = workspace.get(nbytes, K.device)
    elif workspace is None:
        ws = torch.empty(nbytes, dtype=torch.uint8, device=K.device) if nbytes else None
    else:
        ws = workspace
    ws_bytes = 0 if ws is None else ws.numel() * ws.element_size()
    if stream is None:
        stream = torch.cuda.current_stream(K.device)
    st = ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))
    if events is not None:
        arr = (ctypes.c_void_p * len(events))(*[ctypes.c_void_p(e) for e in events])
        rc = lib.flarepp_route_fwd_profiled(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt),
                                            _ptr(K), _ptr(V), float(scale), _ptr(Y), _ptr(ws),
                                            ws_bytes, st, arr, len(events))
        if rc != OK:
            raise FlareppError(rc, "flarepp_route_fwd_profiled")
        return Y
    if debug:
        rc = lib.flarepp_route_fwd_debug(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt),
                                         _ptr(K), _ptr(V), float(scale), _ptr(Y), _ptr(ws),
                                         ws_bytes, st, _ptr(Q_out), _ptr(Z_out))
    else:
        rc = lib.flarepp_route_fwd(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt), _ptr(K),
                                   _ptr(V), float(scale), _ptr(Y), _ptr(ws), ws_bytes, st)
    if rc != OK:
        raise FlareppError(rc, "flarepp_route_fwd" + ("_debug" if debug else ""))
    return Y


def device_status(shape_or_tensors, workspace, stream=None) -> int:
    """The device status word the last call left in ``workspace`` (synchronises ``stream``):
    OK, or ERR_TIMEOUT when a bounded wait inside a kernel gave up."""
    shape = (shape_or_tensors if isinstance(shape_or_tensors, Shape)
             else _shape_of(*shape_or_tensors))
    buf = workspace.buf if isinstance(workspace, Workspace) else workspace
    dev = buf.device if isinstance(buf, torch.Tensor) and buf.is_cuda else None
    with torch.cuda.device(dev):
        if stream is None:
            stream = torch.cuda.current_stream()
        out = ctypes.c_int32(-1)
        rc = load().flarepp_route_device_status(ctypes.byref(shape), _ptr(buf),
                                                ctypes.c_void_p(stream.cuda_stream),
                                                ctypes.byref(out))
    if rc != OK:
        raise FlareppError(rc, "flarepp_route_device_status")
    return int(out.value)


@_on_device("K")
def route_fwd(seeds, Kt, Vt, K, V, scale=None, Y=None, workspace=None, stream=None):
    """Y = routing chain (Sec. 3.2) on device tensors; returns Y [B,H,N,D] (enqueued on
    ``stream``, default torch's current stream)."""
    return _call(False, seeds, Kt, Vt, K, V, scale, Y, workspace, stream, None, None)


class StageEvents:
    """Six timing events the library records around its stages (flarepp_route_fwd_profiled)."""

    def __init__(self, stream=None):
        stream = stream or torch.cuda.current_stream()
        self.events = [torch.cuda.Event(enable_timing=True) for _ in range(N_STAGE_EVENTS)]
        for e in self.events:  # create the underlying cudaEvent_t
            e.record(stream)
        self.handles = [int(e.cuda_event) for e in self.events]

    def stage_ms(self):
        """Milliseconds of each stage of the last recorded call (synchronises on the events)."""
        self.events[-1].synchronize()
        return {name: self.events[i].elapsed_time(self.events[i + 1])
                for i, name in enumerate(STAGES)}


@_on_device("K")
def route_fwd_profiled(seeds, Kt, Vt, K, V, events: StageEvents, scale=None, Y=None,
                       workspace=None, stream=None):
    """``route_fwd`` that records ``events`` around each stage on the launching stream."""
    return _call(False, seeds, Kt, Vt, K, V, scale, Y, workspace, stream, None, None,
                 events.handles)


@_on_device("K")
def route_fwd_noalloc(seeds, Kt, Vt, K, V, scale=None, Y=None, stream=None):
    """``route_fwd`` through flarepp_route_fwd_noalloc: for callers that cannot allocate
    device memory at call time, the library uses its own fixed 64 MiB scratch array instead
    of a workspace (larger shapes raise ERR_WORKSPACE). Calls that overlap on the GPU share
    that array and race; the first call on a device should come before any stream capture.
    Y is allocated here only when not given."""
    lib = load()
    shape = _shape_of(seeds, Kt, Vt, K, V)
    if Y is not None:
        _check_out(Y, K, "Y")
    _check_device("route_fwd_noalloc", K.device, seeds=seeds, Kt=Kt, Vt=Vt, V=V, Y=Y)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y is None:
        Y = torch.empty_like(K)
    if stream is None:
        stream = torch.cuda.current_stream(K.device)
    rc = lib.flarepp_route_fwd_noalloc(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt),
                                       _ptr(K), _ptr(V), float(scale), _ptr(Y),
                                       ctypes.c_void_p(stream.cuda_stream))
    if rc != OK:
        raise FlareppError(rc, "flarepp_route_fwd_noalloc")
    return Y


@_on_device("K")
def route_fwd_debug(seeds, Kt, Vt, K, V, scale=None, Y=None, workspace=None, stream=None):
    """Like ``route_fwd``, also returning the float32 intermediates Q and Z [B,H,M,D]."""
    B, H, N, D = K.shape
    M = seeds.shape[1]
    Q = torch.empty(B, H, M, D, dtype=torch.float32, device=K.device)
    Z = torch.empty_like(Q)
    Y = _call(True, seeds, Kt, Vt, K, V, scale, Y, workspace, stream, Q, Z)
    return Y, Q, Z


@_on_device("K")
def flare_fwd(Q, K, V, scale=None, Y=None, workspace=None, stream=None, Z_out=None):
    """FLARE with learned queries (Sec. 3, eq. prelim_flare_sdpa) on device tensors:
    Z = SDPA(Q_h, K, V), Y = SDPA(K, Q_h, Z). Q [H, M, D] is shared by the batch; K, V
    [B, H, N, D]. Returns Y; ``Z_out`` (float32 [B, H, M, D], device) receives Z if given."""
    lib = load()
    shape = _shape_of(Q, K, V, K, V)
    if Y is not None:
        _check_out(Y, K, "Y")
    if Z_out is not None and (Z_out.dtype != torch.float32 or not Z_out.is_contiguous() or
                              tuple(Z_out.shape) != (shape.B, shape.H, shape.M, shape.D)):
        raise ValueError("Z_out must be a contiguous float32 [B, H, M, D] tensor")
    _check_device("flare_fwd", K.device, Q=Q, V=V, Y=Y, Z_out=Z_out)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y is None:
        Y = torch.empty_like(K)
    nbytes = int(lib.flarepp_route_workspace_bytes(ctypes.byref(shape)))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, K.device)
    st = stream if stream is not None else torch.cuda.current_stream(K.device)
    rc = lib.flarepp_flare_fwd(ctypes.byref(shape), _ptr(Q), _ptr(K), _ptr(V), float(scale),
                               _ptr(Y), None if ws is None else ctypes.c_void_p(ws.data_ptr()),
                               nbytes, ctypes.c_void_p(st.cuda_stream), _ptr(Z_out))
    if rc != OK:
        raise FlareppError(rc, "flarepp_flare_fwd")
    return Y


MIXER_STAGES = ("projection", "chain", "output")


class MixerEvents:
    """Four timing events the library records around the mixer's stages
    (flarepp_mixer_fwd_profiled)."""

    def __init__(self, stream=None):
        stream = stream or torch.cuda.current_stream()
        self.events = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        for e in self.events:  # create the underlying cudaEvent_t
            e.record(stream)
        self.handles = (ctypes.c_void_p * 4)(*[ctypes.c_void_p(int(e.cuda_event))
                                               for e in self.events])

    def stage_ms(self):
        """Milliseconds of each stage of the last recorded call (synchronises on the events)."""
        self.events[-1].synchronize()
        return {s: self.events[i].elapsed_time(self.events[i + 1])
                for i, s in enumerate(MIXER_STAGES)}


@_on_device("X")
def mixer_fwd(X, W_in, Wo, seeds, scale=None, O=None, workspace=None, stream=None, events=None):
    """The FLARE++ mixer layer (Fig. 1) on device tensors: X [B, N, C], W_in [P*C, C] (P = 4:
    K, V, K~, V~; P = 2: shared projection), Wo [C, C] (both out x in), seeds [H, M, D].
    Returns O [B, N, C]."""
    lib = load()
    shape, P = _mixer_shape(X, W_in, Wo, seeds)
    if O is not None:
        _check_out(O, X, "O")
    _check_device("mixer_fwd", X.device, W_in=W_in, Wo=Wo, seeds=seeds, O=O)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if O is None:
        O = torch.empty_like(X)
    nbytes = int(lib.flarepp_mixer_workspace_bytes(ctypes.byref(shape), P))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, X.device)
    st = stream if stream is not None else torch.cuda.current_stream(X.device)
    args = (ctypes.byref(shape), P, _ptr(X), _ptr(W_in), _ptr(Wo), _ptr(seeds), float(scale),
            _ptr(O), None if ws is None else ctypes.c_void_p(ws.data_ptr()), nbytes,
            ctypes.c_void_p(st.cuda_stream))
    if events is None:
        rc = lib.flarepp_mixer_fwd(*args)
    else:
        rc = lib.flarepp_mixer_fwd_profiled(*args, events.handles, 4)
    if rc != OK:
        raise FlareppError(rc, "flarepp_mixer_fwd")
    return O


def _mixer_shape(X, W_in, Wo, seeds):
    for t in (X, W_in, Wo, seeds):
        if not isinstance(t, torch.Tensor) or not t.is_contiguous():
            raise ValueError("inputs must be contiguous torch tensors")
        if t.dtype != torch.bfloat16:
            raise TypeError("the mixer takes bfloat16 tensors")
    if X.dim() != 3 or W_in.dim() != 2 or Wo.dim() != 2 or seeds.dim() != 3:
        raise ValueError("expected X [B,N,C], W_in [P*C,C], Wo [C,C], seeds [H,M,D], C = H*D")
    B, N, C = X.shape
    H, M, D = seeds.shape
    if H * D != C or tuple(Wo.shape) != (C, C) or W_in.shape[1] != C or \
            W_in.shape[0] not in (2 * C, 4 * C):
        raise ValueError("expected X [B,N,C], W_in [P*C,C], Wo [C,C], seeds [H,M,D], C = H*D")
    return make_shape(B, H, N, M, D, torch.bfloat16), W_in.shape[0] // C


@_on_device("X")
def mixer_fwd_train(X, W_in, Wo, seeds, scale=None, O=None, saved=None, workspace=None,
                    stream=None):
    """The mixer layer's forward that keeps its backward's state. Returns (O, saved)."""
    lib = load()
    shape, P = _mixer_shape(X, W_in, Wo, seeds)
    if O is not None:
        _check_out(O, X, "O")
    _check_device("mixer_fwd_train", X.device, W_in=W_in, Wo=Wo, seeds=seeds, O=O, saved=saved)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if O is None:
        O = torch.empty_like(X)
    sbytes = int(lib.flarepp_mixer_saved_bytes(ctypes.byref(shape), P))
    if saved is None or _nbytes(saved) < sbytes:
        saved = torch.empty(max(sbytes, 1), dtype=torch.uint8, device=X.device)
    nbytes = int(lib.flarepp_mixer_workspace_bytes(ctypes.byref(shape), P))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, X.device)
    st = stream if stream is not None else torch.cuda.current_stream(X.device)
    rc = lib.flarepp_mixer_fwd_train(ctypes.byref(shape), P, _ptr(X), _ptr(W_in), _ptr(Wo),
                                     _ptr(seeds), float(scale), _ptr(O), _ptr(saved), sbytes,
                                     None if ws is None else ctypes.c_void_p(ws.data_ptr()),
                                     nbytes, ctypes.c_void_p(st.cuda_stream))
    if rc != OK:
        raise FlareppError(rc, "flarepp_mixer_fwd_train")
    return O, saved


@_on_device("X")
def mixer_bwd(X, W_in, Wo, seeds, saved, dO, scale=None, grads=None, workspace=None,
              stream=None):
    """The mixer layer's backward from :func:`mixer_fwd_train`'s ``saved``: returns
    (dX, dW_in, dWo, dseeds) in bf16; ``grads`` may supply those four output tensors."""
    lib = load()
    shape, P = _mixer_shape(X, W_in, Wo, seeds)
    if tuple(dO.shape) != tuple(X.shape) or dO.dtype != X.dtype or not dO.is_contiguous():
        raise ValueError("dO must be a contiguous tensor of X's shape and dtype")
    if grads is not None:
        if len(grads) != 4:
            raise ValueError("grads must hold four tensors: dX, dW_in, dWo, dseeds")
        grads = tuple(_check_out(g, like, name) for g, like, name in
                      zip(grads, (X, W_in, Wo, seeds), ("dX", "dW_in", "dWo", "dseeds")))
    _check_device("mixer_bwd", X.device, W_in=W_in, Wo=Wo, seeds=seeds, saved=saved, dO=dO,
                  **({} if grads is None else dict(zip(("dX", "dW_in", "dWo", "dseeds"), grads))))
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if grads is None:
        grads = (torch.empty_like(X), torch.empty_like(W_in), torch.empty_like(Wo),
                 torch.empty_like(seeds))
    nbytes = int(lib.flarepp_mixer_bwd_workspace_bytes(ctypes.byref(shape), P))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, X.device)
    st = stream if stream is not None else torch.cuda.current_stream(X.device)
    rc = lib.flarepp_mixer_bwd(ctypes.byref(shape), P, _ptr(X), _ptr(W_in), _ptr(Wo),
                               _ptr(seeds), float(scale), _ptr(saved),
                               _nbytes(saved), _ptr(dO),
                               *(_ptr(g) for g in grads),
                               None if ws is None else ctypes.c_void_p(ws.data_ptr()), nbytes,
                               ctypes.c_void_p(st.cuda_stream))
    if rc != OK:
        raise FlareppError(rc, "flarepp_mixer_bwd")
    return grads


@_on_device("K")
def route_fwd_train(seeds, Kt, Vt, K, V, scale=None, Y=None, saved=None, workspace=None,
                    stream=None):
    """The chain's forward that also keeps the state its backward needs (App. A.5).
    Returns (Y, saved): ``saved`` is an opaque uint8 device tensor for :func:`route_bwd`."""
    lib = load()
    shape = _shape_of(seeds, Kt, Vt, K, V)
    if Y is not None:
        _check_out(Y, K, "Y")
    _check_device("route_fwd_train", K.device, seeds=seeds, Kt=Kt, Vt=Vt, V=V, Y=Y, saved=saved)
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y is None:
        Y = torch.empty_like(K)
    sbytes = int(lib.flarepp_route_saved_bytes(ctypes.byref(shape)))
    if saved is None or _nbytes(saved) < sbytes:
        saved = torch.empty(max(sbytes, 1), dtype=torch.uint8, device=K.device)
    nbytes = int(lib.flarepp_route_workspace_bytes(ctypes.byref(shape)))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, K.device)
    st = stream if stream is not None else torch.cuda.current_stream(K.device)
    rc = lib.flarepp_route_fwd_train(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt),
                                     _ptr(K), _ptr(V), float(scale), _ptr(Y), _ptr(saved),
                                     sbytes, None if ws is None else ctypes.c_void_p(ws.data_ptr()),
                                     nbytes, ctypes.c_void_p(st.cuda_stream))
    if rc != OK:
        raise FlareppError(rc, "flarepp_route_fwd_train")
    return Y, saved


@_on_device("K")
def route_bwd(seeds, Kt, Vt, K, V, Y, dY, saved, scale=None, grads=None, workspace=None,
              stream=None):
    """Backward of the chain (App. A.5) from :func:`route_fwd_train`'s ``Y`` and ``saved``.
    Returns (dseeds [H, M, D], dKt, dVt, dK, dV [B, H, N, D]) in the input dtype; ``grads``
    may supply those five output tensors."""
    lib = load()
    shape = _shape_of(seeds, Kt, Vt, K, V)
    for t in (Y, dY):
        if tuple(t.shape) != tuple(K.shape) or t.dtype != K.dtype or not t.is_contiguous():
            raise ValueError("Y and dY must be contiguous tensors of K's shape and dtype")
    names = ("dseeds", "dKt", "dVt", "dK", "dV")
    if grads is not None:
        if len(grads) != 5:
            raise ValueError("grads must hold five tensors: dseeds, dKt, dVt, dK, dV")
        grads = tuple(_check_out(g, like, name) for g, like, name in
                      zip(grads, (seeds, Kt, Vt, K, V), names))
    _check_device("route_bwd", K.device, seeds=seeds, Kt=Kt, Vt=Vt, V=V, Y=Y, dY=dY,
                  saved=saved, **({} if grads is None else dict(zip(names, grads))))
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if grads is None:
        grads = (torch.empty_like(seeds), torch.empty_like(Kt), torch.empty_like(Vt),
                 torch.empty_like(K), torch.empty_like(V))
    sbytes = int(lib.flarepp_route_saved_bytes(ctypes.byref(shape)))
    nbytes = int(lib.flarepp_route_bwd_workspace_bytes(ctypes.byref(shape)))
    ws = (workspace if isinstance(workspace, Workspace) else Workspace()).get(nbytes, K.device)
    st = stream if stream is not None else torch.cuda.current_stream(K.device)
    rc = lib.flarepp_route_bwd(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt), _ptr(K),
                               _ptr(V), float(scale), _ptr(Y), _ptr(dY), _ptr(saved),
                               _nbytes(saved),
                               *(_ptr(g) for g in grads),
                               None if ws is None else ctypes.c_void_p(ws.data_ptr()), nbytes,
                               ctypes.c_void_p(st.cuda_stream))
    if rc != OK:
        raise FlareppError(rc, "flarepp_route_bwd")
    return grads


@_on_device("device")
def route_fwd_host(seeds, Kt, Vt, K, V, scale=None, Y_host=None, device="cuda", workspace=None,
                   stream=None, dev_bufs=None):
    """End-to-end call on host tensors through ``flarepp_route_fwd_host``: the library copies
    the inputs to the device, runs the chain and copies Y back into ``Y_host`` (allocated
    pinned here if not given), overlapping the copies with the computation by head groups.
    Pass pinned host tensors for the copies to overlap. Returns Y_host once the copy has
    completed. ``workspace`` (a :class:`Workspace`) holds the device buffer between calls;
    ``dev_bufs`` is accepted for compatibility and unused."""
    del dev_bufs
    lib = load()
    shape = _shape_of(seeds, Kt, Vt, K, V)
    for t in (seeds, Kt, Vt, K, V):
        if t.is_cuda:
            raise ValueError("route_fwd_host takes host tensors")
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y_host is None:
        Y_host = torch.empty(K.shape, dtype=K.dtype, pin_memory=True)
    elif tuple(Y_host.shape) != tuple(K.shape) or Y_host.dtype != K.dtype or Y_host.is_cuda:
        raise ValueError("Y_host must be a host tensor of K's shape and dtype")
    dev = torch.device(device)
    if dev.index is None:
        dev = torch.device("cuda", torch.cuda.current_device())
    nbytes = int(lib.flarepp_route_host_buffer_bytes(ctypes.byref(shape)))
    ws = workspace if workspace is not None else Workspace()
    buf = ws.get(nbytes, dev) if nbytes else None
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    rc = lib.flarepp_route_fwd_host(ctypes.byref(shape), _ptr(seeds), _ptr(Kt), _ptr(Vt), _ptr(K),
                                    _ptr(V), float(scale), _ptr(Y_host),
                                    None if buf is None else ctypes.c_void_p(buf.data_ptr()),
                                    nbytes, ctypes.c_void_p(st.cuda_stream))
    if rc != 0:
        raise FlareppError(rc, "flarepp_route_fwd_host")
    st.synchronize()
    return Y_host


@_on_device("device")
def flare_fwd_host(Q, K, V, scale=None, Y_host=None, device="cuda", workspace=None, stream=None):
    """FLARE with learned queries Q [H, M, D] on host tensors through
    ``flarepp_flare_fwd_host``: copies in, FLARE, Y copied back into ``Y_host`` (allocated
    pinned here if not given), overlapped by head groups. Returns Y_host once it is filled."""
    lib = load()
    shape = _shape_of(Q, K, V, K, V)
    for t in (Q, K, V):
        if t.is_cuda:
            raise ValueError("flare_fwd_host takes host tensors")
    if scale is None:
        scale = 1.0 / math.sqrt(shape.D)
    if Y_host is None:
        Y_host = torch.empty(K.shape, dtype=K.dtype, pin_memory=True)
    elif tuple(Y_host.shape) != tuple(K.shape) or Y_host.dtype != K.dtype or Y_host.is_cuda:
        raise ValueError("Y_host must be a host tensor of K's shape and dtype")
    dev = torch.device(device)
    if dev.index is None:
        dev = torch.device("cuda", torch.cuda.current_device())
    nbytes = int(lib.flarepp_route_host_buffer_bytes(ctypes.byref(shape)))
    ws = workspace if workspace is not None else Workspace()
    buf = ws.get(nbytes, dev) if nbytes else None
    st = stream if stream is not None else torch.cuda.current_stream(dev)
    rc = lib.flarepp_flare_fwd_host(ctypes.byref(shape), _ptr(Q), _ptr(K), _ptr(V),
                                    float(scale), _ptr(Y_host),
                                    None if buf is None else ctypes.c_void_p(buf.data_ptr()),
                                    nbytes, ctypes.c_void_p(st.cuda_stream))
    if rc != 0:
        raise FlareppError(rc, "flarepp_flare_fwd_host")
    st.synchronize()
    return Y_host
