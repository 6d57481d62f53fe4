"""Python binding of the MoCE C ABI (include/moce.h).

Argument marshalling only: every step of the layer runs in the CUDA kernels
of ``libmoce.so``. PyTorch provides device memory and the current stream.
There is no CPU fallback: if the library is not built, or a tensor is not on
a CUDA device, the call raises.

The functions carry the C names. Tensors:
  x              NHWC [N, H, W, C_in] or NCHW [N, C_in, H, W]; torch.bfloat16 or float32
  y              same layout/dtype with C_out + 1 channels (residual expert last)
  support_idx    int32 [C_out, k]; support_logits float32 [C_out, k]
  W1 [k, k] (row j = hidden unit j), b1 [k], w2 [k], b2 [1]: float32
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from . import build as _build

MOCE_OK, MOCE_ERR_INVALID_VALUE, MOCE_ERR_BAD_SUPPORT = 0, 1, 2
MOCE_ERR_UNSUPPORTED, MOCE_ERR_CUDA, MOCE_ERR_TIMEOUT = 3, 4, 5
MOCE_F32, MOCE_BF16 = 0, 1
MOCE_NHWC, MOCE_NCHW = 0, 1
_LAYOUTS = {"nhwc": MOCE_NHWC, "nchw": MOCE_NCHW}

_lib = None


class MoceError(RuntimeError):
    def __init__(self, status: int, what: str):
        name = library().moce_status_string(status).decode()
        super().__init__(f"{what} failed: {name}")
        self.status = status


def library_path() -> str:
    return _build.LIB


def library():
    """The loaded ``libmoce.so`` (raises if it has not been built)."""
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            raise RuntimeError(f"MoCE CUDA library not built ({path}); run "
                               "paper_2608_23794_gb300.build.build() first")
        lib = ctypes.CDLL(path)
        P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        sig = {
            "moce_status_string": ([I], ctypes.c_char_p),
            "moce_pack_workspace_bytes": ([I, I, I], S),
            "moce_pack_supports": ([I, I, I, P, P, P, P, P, P, P, S, P], I),
            "moce_workspace_bytes": ([I, I, I, I, I, I], S),
            "moce_workspace_init": ([P, S, P], I),
            "moce_workspace_offsets": ([I, I, I, I, I, I, P, P], I),
            "moce_pool": ([P, I, I, I, I, I, I, P, P, S, P], I),
            "moce_gate": ([P, I, I, I, I, P, P, P, P, P, P, F, F, P, P, P], I),
            "moce_forward": ([P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F, P, P, S, P], I),
            "moce_forward_path": ([P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F, P, P, S,
                                   I, P], I),
            "moce_forward_path_launches": ([P, I, I, I, I, I, I, I, I, I], I),
            "moce_forward_path_kernel": ([P, I, I, I, I, I, I, I, I, I], ctypes.c_char_p),
            "moce_check_device_error": ([P, S, P], I),
            "moce_forward_launches": ([P, I, I, I, I, I, I, I, I], I),
            "moce_forward_kernel": ([P, I, I, I, I, I, I, I, I], ctypes.c_char_p),
            "moce_forward_noalloc": ([P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F, P, P], I),
            "moce_noalloc_check_device_error": ([P], I),
            "moce_train_workspace_bytes": ([I, I], S),
            "moce_topk_supports": ([P, I, I, I, P, P, P, S, P], I),
            "moce_coverage_loss": ([P, I, I, F, P, P, P, P, S, P], I),
            "moce_backward_workspace_bytes": ([I, I, I, I, I, I], S),
            "moce_mix": ([P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, S, P], I),
            "moce_dynamic_workspace_bytes": ([I, I, I, I, I, I, I], S),
            "moce_dynamic_supports": ([P, I, I, I, I, I, P, P, P, P, P, P, P, P, P, P, S, P], I),
            "moce_forward_supports": ([P, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, P, F, F, P,
                                       P, S, P], I),
            "moce_forward_dynamic": ([P, I, I, I, I, I, I, I, I, I, P, P, P, P, P, P, P, P, P, F, F,
                                      P, P, P, P, P, S, P], I),
            "moce_backward": ([P, P, I, I, I, I, I, I, I, I, P, P, P, I, P, P, P, P, F, F,
                               P, P, P, P, P, P, P, S, P], I),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes, fn.restype = args, res
        _lib = lib
    return _lib


def _check(status: int, what: str):
    if status != MOCE_OK:
        raise MoceError(status, what)


def _ptr(t: torch.Tensor | None):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("MoCE tensors must be CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("MoCE tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream: torch.cuda.Stream | None = None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return MOCE_BF16
    if t.dtype == torch.float32:
        return MOCE_F32
    raise ValueError(f"unsupported dtype {t.dtype}")


def _dims(x: torch.Tensor, layout: str):
    if layout == "nhwc":
        N, H, W, C = x.shape
    elif layout == "nchw":
        N, C, H, W = x.shape
    else:
        raise ValueError(layout)
    return N, H, W, C


@dataclass
class PackedSupports:
    packed_idx: torch.Tensor      # int32 [C_out, k], rows in deployment order
    packed_logits: torch.Tensor   # float32 [C_out, k]
    resid_idx: torch.Tensor       # int32 [C_in]; the first n_resid entries are U
    n_resid: int
    C_in: int

    @property
    def C_out(self) -> int:
        return self.packed_idx.shape[0]

    @property
    def k(self) -> int:
        return self.packed_idx.shape[1]


def moce_pack_supports(support_idx: torch.Tensor, support_logits: torch.Tensor, C_in: int,
                       stream=None) -> PackedSupports:
    R, k = support_idx.shape
    dev = support_idx.device
    out_idx = torch.empty((R, k), dtype=torch.int32, device=dev)
    out_lg = torch.empty((R, k), dtype=torch.float32, device=dev)
    resid = torch.empty((C_in,), dtype=torch.int32, device=dev)
    ws_bytes = library().moce_pack_workspace_bytes(C_in, R, k)
    if ws_bytes == 0:
        raise MoceError(MOCE_ERR_INVALID_VALUE, "moce_pack_workspace_bytes")
    ws = torch.empty((ws_bytes,), dtype=torch.uint8, device=dev)
    n_resid = ctypes.c_int32(0)
    _check(library().moce_pack_supports(C_in, R, k, _ptr(support_idx.to(torch.int32).contiguous()),
                                        _ptr(support_logits.to(torch.float32).contiguous()),
                                        _ptr(out_idx), _ptr(out_lg), _ptr(resid),
                                        ctypes.byref(n_resid), _ptr(ws), ws_bytes, _stream(stream)),
           "moce_pack_supports")
    return PackedSupports(out_idx, out_lg, resid, int(n_resid.value), C_in)


def moce_status_string(status: int) -> str:
    return library().moce_status_string(int(status)).decode()


def moce_pack_workspace_bytes(C_in: int, C_out: int, k: int) -> int:
    return int(library().moce_pack_workspace_bytes(C_in, C_out, k))


def moce_workspace_bytes(N: int, H: int, W: int, C_in: int, C_out: int, k: int) -> int:
    return int(library().moce_workspace_bytes(N, H, W, C_in, C_out, k))


def moce_workspace_offsets(N: int, H: int, W: int, C_in: int, C_out: int, k: int):
    """Byte offsets of z and tau inside the forward workspace of this shape."""
    z_off, tau_off = ctypes.c_size_t(0), ctypes.c_size_t(0)
    _check(library().moce_workspace_offsets(N, H, W, C_in, C_out, k, ctypes.byref(z_off),
                                            ctypes.byref(tau_off)), "moce_workspace_offsets")
    return z_off.value, tau_off.value


class Workspace:
    """A zero-initialised forward workspace for one layer shape."""

    def __init__(self, N, H, W, C_in, C_out, k, device="cuda"):
        self.shape = (N, H, W, C_in, C_out, k)
        nbytes = moce_workspace_bytes(N, H, W, C_in, C_out, k)
        if nbytes == 0:
            raise MoceError(MOCE_ERR_INVALID_VALUE, "moce_workspace_bytes")
        self.buffer = torch.zeros((nbytes,), dtype=torch.uint8, device=device)
        self.z_offset, self.tau_offset = moce_workspace_offsets(N, H, W, C_in, C_out, k)

    @property
    def nbytes(self) -> int:
        return self.buffer.numel()

    def z(self) -> torch.Tensor:
        N, _, _, C, _, _ = self.shape
        return self.buffer[self.z_offset:self.z_offset + 4 * N * C].view(torch.float32).view(N, C)

    def tau(self) -> torch.Tensor:
        N, _, _, _, R, _ = self.shape
        return self.buffer[self.tau_offset:self.tau_offset + 4 * N * R].view(torch.float32).view(N, R)

    def init(self, stream=None):
        moce_workspace_init(self, stream)


def moce_workspace_init(ws: Workspace, stream=None):
    """Zero-fill a forward workspace on the stream (needed again after MOCE_ERR_TIMEOUT)."""
    _check(library().moce_workspace_init(_ptr(ws.buffer), ws.nbytes, _stream(stream)),
           "moce_workspace_init")


def moce_pool(x: torch.Tensor, layout: str, ws: Workspace | None = None, z=None,
              stream=None) -> torch.Tensor:
    N, H, W, C = _dims(x, layout)
    if z is None:
        z = torch.empty((N, C), dtype=torch.float32, device=x.device)
    if ws is None:
        ws = Workspace(N, H, W, C, 1, 1, device=x.device)
    _check(library().moce_pool(_ptr(x), N, H, W, C, _dtype(x), _LAYOUTS[layout], _ptr(z),
                               _ptr(ws.buffer), ws.nbytes, _stream(stream)), "moce_pool")
    return z


def moce_gate(z: torch.Tensor, packed: PackedSupports, W1, b1, w2, b2, tau_min: float,
              tau_max: float, want_weights: bool = True, stream=None):
    N, C = z.shape
    R, k = packed.C_out, packed.k
    tau = torch.empty((N, R), dtype=torch.float32, device=z.device)
    a = torch.empty((N, R, k), dtype=torch.float32, device=z.device) if want_weights else None
    _check(library().moce_gate(_ptr(z), N, C, R, k, _ptr(packed.packed_idx),
                               _ptr(packed.packed_logits), _ptr(W1), _ptr(b1), _ptr(w2), _ptr(b2),
                               float(tau_min), float(tau_max), _ptr(tau), _ptr(a),
                               _stream(stream)), "moce_gate")
    return tau, a


# moce_path_t: the kernel path of one forward (AUTO = the fastest that fits)
PATHS = {"auto": 0, "steps": 4, "stream": 6}


def moce_forward(x: torch.Tensor, layout: str, packed: PackedSupports, W1, b1, w2, b2,
                 tau_min: float, tau_max: float, ws: Workspace | None = None,
                 y: torch.Tensor | None = None, stream=None, path: str = "auto") -> torch.Tensor:
    """The layer forward (Sec. 3.2-3.4); ``path`` forces one kernel path (``PATHS``)."""
    N, H, W, C = _dims(x, layout)
    R, k = packed.C_out, packed.k
    if C != packed.C_in:
        raise ValueError("x channels do not match the packed supports")
    if y is None:
        shape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
        y = torch.empty(shape, dtype=x.dtype, device=x.device)
    if ws is None:
        ws = Workspace(N, H, W, C, R, k, device=x.device)
    lib = library()
    args = (_ptr(x), N, H, W, C, R, k, _dtype(x), _LAYOUTS[layout], _ptr(packed.packed_idx),
            _ptr(packed.packed_logits), _ptr(packed.resid_idx), packed.n_resid, _ptr(W1), _ptr(b1),
            _ptr(w2), _ptr(b2), float(tau_min), float(tau_max), _ptr(y), _ptr(ws.buffer), ws.nbytes)
    if path == "auto":
        _check(lib.moce_forward(*args, _stream(stream)), "moce_forward")
    else:
        _check(lib.moce_forward_path(*args, PATHS[path], _stream(stream)), "moce_forward_path")
    return y


def moce_forward_path(x: torch.Tensor, layout: str, packed: PackedSupports, W1, b1, w2, b2,
                      tau_min: float, tau_max: float, path: str, ws: Workspace | None = None,
                      y: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """moce_forward on the kernel path ``path`` (a key of ``PATHS``)."""
    return moce_forward(x, layout, packed, W1, b1, w2, b2, tau_min, tau_max, ws=ws, y=y,
                        stream=stream, path=path)


def moce_forward_path_launches(x: torch.Tensor, layout: str, C_out: int, k: int, path: str) -> int:
    return moce_forward_launches(x, layout, C_out, k, path=path)


def moce_forward_path_kernel(x: torch.Tensor, layout: str, C_out: int, k: int, path: str) -> str:
    return moce_forward_kernel(x, layout, C_out, k, path=path)


def moce_forward_launches(x: torch.Tensor, layout: str, C_out: int, k: int,
                          path: str = "auto") -> int:
    """Kernel launches one moce_forward call makes for this input (0: path cannot run it)."""
    N, H, W, C = _dims(x, layout)
    if path == "auto":
        return int(library().moce_forward_launches(_ptr(x), N, H, W, C, C_out, k, _dtype(x),
                                                    _LAYOUTS[layout]))
    return int(library().moce_forward_path_launches(_ptr(x), N, H, W, C, C_out, k, _dtype(x),
                                                     _LAYOUTS[layout], PATHS[path]))


def moce_forward_kernel(x: torch.Tensor, layout: str, C_out: int, k: int,
                        path: str = "auto") -> str:
    """Name of the kernel path one moce_forward call takes for this input."""
    N, H, W, C = _dims(x, layout)
    if path == "auto":
        name = library().moce_forward_kernel(_ptr(x), N, H, W, C, C_out, k, _dtype(x),
                                             _LAYOUTS[layout])
    else:
        name = library().moce_forward_path_kernel(_ptr(x), N, H, W, C, C_out, k, _dtype(x),
                                                  _LAYOUTS[layout], PATHS[path])
    if name is None:
        raise MoceError(1, "moce_forward_kernel")
    return name.decode()


def moce_forward_noalloc(x: torch.Tensor, layout: str, packed: PackedSupports, W1, b1, w2, b2,
                         tau_min: float, tau_max: float, y: torch.Tensor | None = None,
                         stream=None) -> torch.Tensor:
    """moce_forward without a workspace, for callers that cannot allocate device memory.

    The scratch is a fixed array inside the library (8 MiB per device); layers
    that need more are rejected. Calls that overlap on the GPU share it and race.
    """
    N, H, W, C = _dims(x, layout)
    R, k = packed.C_out, packed.k
    if C != packed.C_in:
        raise ValueError("x channels do not match the packed supports")
    if y is None:
        shape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
        y = torch.empty(shape, dtype=x.dtype, device=x.device)
    _check(library().moce_forward_noalloc(_ptr(x), N, H, W, C, R, k, _dtype(x), _LAYOUTS[layout],
                                          _ptr(packed.packed_idx), _ptr(packed.packed_logits),
                                          _ptr(packed.resid_idx), packed.n_resid, _ptr(W1),
                                          _ptr(b1), _ptr(w2), _ptr(b2), float(tau_min),
                                          float(tau_max), _ptr(y), _stream(stream)),
           "moce_forward_noalloc")
    return y


def moce_train_workspace_bytes(C_in: int, C_out: int) -> int:
    return int(library().moce_train_workspace_bytes(C_in, C_out))


def _train_ws(C_in: int, C_out: int, device) -> torch.Tensor:
    nbytes = library().moce_train_workspace_bytes(C_in, C_out)
    if nbytes == 0:
        raise MoceError(MOCE_ERR_INVALID_VALUE, "moce_train_workspace_bytes")
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def moce_topk_supports(logits: torch.Tensor, k: int, stream=None):
    """Eq. (support): the top-k channels of each row of logits [C_out, C_in], in deployment order.

    Returns (packed_idx int32 [C_out, k], packed_logits float32 [C_out, k]). Synchronous.
    """
    logits = logits.contiguous()
    if logits.dtype != torch.float32 or logits.dim() != 2:
        raise ValueError("logits must be float32 [C_out, C_in]")
    R, C = logits.shape
    idx = torch.empty((R, k), dtype=torch.int32, device=logits.device)
    lg = torch.empty((R, k), dtype=torch.float32, device=logits.device)
    ws = _train_ws(C, R, logits.device)
    _check(library().moce_topk_supports(_ptr(logits), C, R, k, _ptr(idx), _ptr(lg), _ptr(ws),
                                        ws.numel(), _stream(stream)), "moce_topk_supports")
    return idx, lg


def moce_coverage_loss(logits: torch.Tensor, eps: float, grad: bool = True, stream=None):
    """Sec. 3.4 coverage regularizer: (loss [1], usage u [C_in], dloss/dlogits [C_out, C_in] or None)."""
    logits = logits.contiguous()
    if logits.dtype != torch.float32 or logits.dim() != 2:
        raise ValueError("logits must be float32 [C_out, C_in]")
    R, C = logits.shape
    loss = torch.empty(1, dtype=torch.float32, device=logits.device)
    usage = torch.empty(C, dtype=torch.float32, device=logits.device)
    g = torch.empty((R, C), dtype=torch.float32, device=logits.device) if grad else None
    ws = _train_ws(C, R, logits.device)
    _check(library().moce_coverage_loss(_ptr(logits), C, R, float(eps), _ptr(loss), _ptr(usage),
                                        _ptr(g) if g is not None else None, _ptr(ws), ws.numel(),
                                        _stream(stream)), "moce_coverage_loss")
    return loss, usage, g


@dataclass
class Gradients:
    dx: torch.Tensor        # float32, the shape and layout of x
    dlogits: torch.Tensor   # float32 [C_out, k], packed order
    dW1: torch.Tensor       # float32 [k, k]
    db1: torch.Tensor       # float32 [k]
    dw2: torch.Tensor       # float32 [k]
    db2: torch.Tensor       # float32 [1]


def moce_backward_workspace_bytes(N: int, H: int, W: int, C_in: int, C_out: int, k: int) -> int:
    return int(library().moce_backward_workspace_bytes(N, H, W, C_in, C_out, k))


def moce_backward(x: torch.Tensor, dy: torch.Tensor, layout: str, packed: PackedSupports, W1, b1,
                  w2, b2, tau_min: float, tau_max: float, ws: torch.Tensor | None = None,
                  out: Gradients | None = None, stream=None) -> Gradients:
    """Gradients of the layer with static supports for the upstream gradient dy (Sec. 3.2).

    ``out`` (optional) receives the gradients in place; every field is overwritten."""
    N, H, W, C = _dims(x, layout)
    R, k = packed.C_out, packed.k
    if C != packed.C_in:
        raise ValueError("x channels do not match the packed supports")
    if dy.dtype != x.dtype or tuple(_dims(dy, layout)) != (N, H, W, R + 1):
        raise ValueError("dy must have the dtype of x and the shape of y")
    dev = x.device
    f32 = dict(dtype=torch.float32, device=dev)
    g = out or Gradients(torch.empty(x.shape, **f32), torch.empty((R, k), **f32),
                         torch.empty((k, k), **f32), torch.empty(k, **f32), torch.empty(k, **f32),
                         torch.empty(1, **f32))
    if tuple(g.dx.shape) != tuple(x.shape) or g.dlogits.shape != (R, k) or g.dW1.shape != (k, k):
        raise ValueError("gradient buffers do not match the layer")
    if ws is None:
        nbytes = moce_backward_workspace_bytes(N, H, W, C, R, k)
        if nbytes == 0:
            raise MoceError(MOCE_ERR_UNSUPPORTED, "moce_backward_workspace_bytes")
        ws = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    _check(library().moce_backward(_ptr(x), _ptr(dy), N, H, W, C, R, k, _dtype(x),
                                   _LAYOUTS[layout], _ptr(packed.packed_idx),
                                   _ptr(packed.packed_logits), _ptr(packed.resid_idx),
                                   packed.n_resid, _ptr(W1), _ptr(b1), _ptr(w2), _ptr(b2),
                                   float(tau_min), float(tau_max), _ptr(g.dx), _ptr(g.dlogits),
                                   _ptr(g.dW1), _ptr(g.db1), _ptr(g.dw2), _ptr(g.db2), _ptr(ws),
                                   ws.numel(), _stream(stream)), "moce_backward")
    return g


def moce_mix(x: torch.Tensor, layout: str, sup_idx: torch.Tensor, mix_w: torch.Tensor,
             resid_idx: torch.Tensor, n_resid, ws: Workspace, y: torch.Tensor | None = None,
             stream=None) -> torch.Tensor:
    """Eq. (expert) and Eq. (res) from weights mix_w [N, C_out, k].

    Shared supports: sup_idx [C_out, k], resid_idx [C_in], n_resid an int. Per-example
    supports: sup_idx [N, C_out, k], resid_idx [N, C_in], n_resid an int32 CUDA tensor [N].
    """
    N, H, W, C = _dims(x, layout)
    R, k = sup_idx.shape[-2], sup_idx.shape[-1]
    if y is None:
        shape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
        y = torch.empty(shape, dtype=x.dtype, device=x.device)
    per = isinstance(n_resid, torch.Tensor)
    _check(library().moce_mix(_ptr(x), N, H, W, C, R, k, _dtype(x), _LAYOUTS[layout],
                              _ptr(sup_idx), _ptr(mix_w), _ptr(resid_idx),
                              0 if per else int(n_resid), _ptr(n_resid) if per else None, _ptr(y),
                              _ptr(ws.buffer), ws.nbytes, _stream(stream)), "moce_mix")
    return y


@dataclass
class DynamicRouter:
    """Parameters of Eq. (dynamic): the static routing matrix and the rank-d router."""
    logits: torch.Tensor   # float32 [C_out, C_in]
    Wh: torch.Tensor       # float32 [d, C_in]
    bh: torch.Tensor       # float32 [d]
    V: torch.Tensor        # float32 [C_in, d], row c = v_c
    Q: torch.Tensor        # float32 [C_out, d], row e = q_e

    @property
    def d(self) -> int:
        return self.Wh.shape[0]


@dataclass
class DynamicSupports:
    sup_idx: torch.Tensor     # int32 [N, C_out, k], deployment order per example
    sup_logits: torch.Tensor  # float32 [N, C_out, k]: the selected L_e(X) values
    resid_idx: torch.Tensor   # int32 [N, C_in]: row n starts with U(X) ascending
    n_resid: torch.Tensor     # int32 [N]


def moce_dynamic_workspace_bytes(N, H, W, C_in, C_out, k, d) -> int:
    return int(library().moce_dynamic_workspace_bytes(N, H, W, C_in, C_out, k, d))


def _dyn_ws(N, H, W, C, R, k, d, device):
    nbytes = moce_dynamic_workspace_bytes(N, H, W, C, R, k, d)
    if nbytes == 0:
        raise MoceError(MOCE_ERR_UNSUPPORTED, "moce_dynamic_workspace_bytes")
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def _empty_supports(N, R, k, C, device) -> DynamicSupports:
    return DynamicSupports(torch.empty((N, R, k), dtype=torch.int32, device=device),
                           torch.empty((N, R, k), dtype=torch.float32, device=device),
                           torch.empty((N, C), dtype=torch.int32, device=device),
                           torch.empty(N, dtype=torch.int32, device=device))


def moce_dynamic_supports(z: torch.Tensor, router: DynamicRouter, k: int,
                          ws: torch.Tensor | None = None, out: DynamicSupports | None = None,
                          stream=None) -> DynamicSupports:
    """Per-example supports of Eq. (dynamic) from pooled descriptors z [N, C_in]."""
    N, C = z.shape
    R, d = router.logits.shape[0], router.d
    sup = out or _empty_supports(N, R, k, C, z.device)
    if ws is None:
        ws = _dyn_ws(N, 1, 1, C, R, k, d, z.device)
    _check(library().moce_dynamic_supports(_ptr(z), N, C, R, k, d, _ptr(router.logits),
                                           _ptr(router.Wh), _ptr(router.bh), _ptr(router.V),
                                           _ptr(router.Q), _ptr(sup.sup_idx), _ptr(sup.sup_logits),
                                           _ptr(sup.resid_idx), _ptr(sup.n_resid), _ptr(ws),
                                           ws.numel(), _stream(stream)), "moce_dynamic_supports")
    return sup


def moce_forward_supports(x: torch.Tensor, layout: str, sup: DynamicSupports, W1, b1, w2, b2,
                          tau_min: float, tau_max: float, ws: Workspace | None = None,
                          y: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """The layer with given per-example supports (pool, gate, mix)."""
    N, H, W, C = _dims(x, layout)
    R, k = sup.sup_idx.shape[1], sup.sup_idx.shape[2]
    if y is None:
        shape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
        y = torch.empty(shape, dtype=x.dtype, device=x.device)
    if ws is None:
        ws = Workspace(N, H, W, C, R, k, device=x.device)
    _check(library().moce_forward_supports(_ptr(x), N, H, W, C, R, k, _dtype(x), _LAYOUTS[layout],
                                           _ptr(sup.sup_idx), _ptr(sup.sup_logits),
                                           _ptr(sup.resid_idx), _ptr(sup.n_resid), _ptr(W1),
                                           _ptr(b1), _ptr(w2), _ptr(b2), float(tau_min),
                                           float(tau_max), _ptr(y), _ptr(ws.buffer), ws.nbytes,
                                           _stream(stream)), "moce_forward_supports")
    return y


def moce_forward_dynamic(x: torch.Tensor, layout: str, router: DynamicRouter, k: int, W1, b1, w2,
                         b2, tau_min: float, tau_max: float, ws: torch.Tensor | None = None,
                         y: torch.Tensor | None = None, supports: DynamicSupports | None = None,
                         stream=None) -> torch.Tensor:
    """The input-conditioned support variant (Eq. dynamic), inference path.

    ``supports`` (optional) receives the per-example supports and |U(X)|; its resid_idx is
    not written (U(X) stays in the workspace).
    """
    N, H, W, C = _dims(x, layout)
    R, d = router.logits.shape[0], router.d
    if y is None:
        shape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
        y = torch.empty(shape, dtype=x.dtype, device=x.device)
    if ws is None:
        ws = _dyn_ws(N, H, W, C, R, k, d, x.device)
    _check(library().moce_forward_dynamic(
        _ptr(x), N, H, W, C, R, k, d, _dtype(x), _LAYOUTS[layout], _ptr(router.logits),
        _ptr(router.Wh), _ptr(router.bh), _ptr(router.V), _ptr(router.Q), _ptr(W1), _ptr(b1),
        _ptr(w2), _ptr(b2), float(tau_min), float(tau_max), _ptr(y),
        _ptr(supports.sup_idx) if supports else None,
        _ptr(supports.sup_logits) if supports else None,
        _ptr(supports.n_resid) if supports else None, _ptr(ws), ws.numel(), _stream(stream)),
        "moce_forward_dynamic")
    return y


def moce_noalloc_check_device_error(stream=None):
    """Raise if a bounded wait of the last moce_forward_noalloc on this device gave up (synchronous)."""
    _check(library().moce_noalloc_check_device_error(_stream(stream)),
           "moce_noalloc_check_device_error")


def moce_check_device_error(ws: Workspace, stream=None):
    _check(library().moce_check_device_error(_ptr(ws.buffer), ws.nbytes, _stream(stream)),
           "moce_check_device_error")
