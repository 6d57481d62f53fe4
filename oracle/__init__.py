"""CPU oracle for the MoCE layer forward (test infrastructure only).

A ctypes wrapper around ``moce_oracle.c``: a plain double-precision restatement
of the layer of "Mixture of Channel Experts" (Sec. 3, Eqs. support, tau,
weights, expert, res). Only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg may import this package. The CUDA
library never imports it and shares no code with it.

Every function takes and returns numpy arrays. ``x`` is passed as float32
holding exactly the values the device sees (bf16 inputs decoded to float32).
Layouts: ``"nhwc"`` (channel fastest) or ``"nchw"`` (pixel fastest); ``y`` has
``R + 1`` channels in the layout of ``x``, the residual expert last.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "moce_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libmoce_oracle.so")

OK, BAD_ARG, BAD_SUPPORT, NO_MEMORY = 0, 1, 2, 3
_LAYOUT = {"nhwc": 0, "nchw": 1}

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into ``oracle/_build/libmoce_oracle.so``."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        F = ctypes.c_float
        D = ctypes.c_double
        lib.moce_oracle_topk.argtypes = [I, I, I, P, P, P]
        lib.moce_oracle_pack.argtypes = [I, I, I, P, P, P, P, P, P]
        lib.moce_oracle_pool.argtypes = [P, I, I, I, I, I, P]
        lib.moce_oracle_pool.restype = None
        lib.moce_oracle_gate.argtypes = [P, I, I, I, I, P, P, P, P, F, D, D, P, P]
        lib.moce_oracle_gate.restype = None
        lib.moce_oracle_weights.argtypes = [P, I, I, I, P, P]
        lib.moce_oracle_weights.restype = None
        lib.moce_oracle_mix.argtypes = [P, I, I, I, I, I, I, I, P, P, P, I, P]
        lib.moce_oracle_mix.restype = None
        lib.moce_oracle_forward.argtypes = [P, I, I, I, I, I, I, I, P, P, P, I, P, P, P, F, D, D,
                                            P, P, P, P]
        lib.moce_oracle_bruteforce_forward.argtypes = [P, I, I, I, I, I, I, I, P, P, P, P, F, D, D,
                                                       P]
        lib.moce_oracle_coverage.argtypes = [I, I, P, D, P, P, P]
        lib.moce_oracle_backward.argtypes = [P, P, I, I, I, I, I, I, I, P, P, P, I, P, P, P, F, D,
                                             D, P, P, P, P, P, P]
        lib.moce_oracle_dynamic_logits.argtypes = [P, I, I, I, I, I, I, I, P, P, P, P, P, P, P]
        for fn in (lib.moce_oracle_topk, lib.moce_oracle_pack, lib.moce_oracle_forward,
                   lib.moce_oracle_bruteforce_forward, lib.moce_oracle_coverage,
                   lib.moce_oracle_backward, lib.moce_oracle_dynamic_logits):
            fn.restype = ctypes.c_int
        _lib = lib
    return _lib


class OracleError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: oracle status {status}")
        self.status = status


def _c(a: np.ndarray, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def _p(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def topk(L: np.ndarray, k: int):
    """Eq. (support): the k largest logits of each row of L [R, C], in deployment order."""
    L = _c(L, np.float32)
    R, C = L.shape
    idx = np.empty((R, k), np.int32)
    lg = np.empty((R, k), np.float32)
    st = _load().moce_oracle_topk(C, R, k, _p(L), _p(idx), _p(lg))
    if st != OK:
        raise OracleError(st, "topk")
    return idx, lg


def coverage(L: np.ndarray, eps: float, grad: bool = True):
    """Sec. 3.4 coverage regularizer over the full routing matrix L [R, C].

    Returns (loss, u [C], dloss/dL [R, C] or None), all float64.
    """
    L = _c(L, np.float32)
    R, C = L.shape
    loss = np.zeros(1, np.float64)
    u = np.empty(C, np.float64)
    g = np.empty((R, C), np.float64) if grad else None
    st = _load().moce_oracle_coverage(C, R, _p(L), float(eps), _p(loss), _p(u), _p(g))
    if st != OK:
        raise OracleError(st, "coverage")
    return float(loss[0]), u, g


def backward(x: np.ndarray, dy: np.ndarray, layout: str, packed_idx, packed_logits, resid, W1,
             b1, w2, b2: float, tau_min: float, tau_max: float):
    """Gradients of the layer (static supports, Sec. 3.2) for the upstream gradient dy.

    Returns a dict of float64 arrays: dx (the shape of x), dlogit [R, k], dW1 [k, k],
    db1 [k], dw2 [k], db2 (float).
    """
    x = _c(x, np.float32)
    dy = _c(dy, np.float32)
    if layout == "nhwc":
        N, H, W, C = x.shape
    else:
        N, C, H, W = x.shape
    pidx = _c(packed_idx, np.int32)
    R, k = pidx.shape
    plog = _c(packed_logits, np.float32)
    resid = _c(resid, np.int32)
    W1 = _c(W1, np.float32)
    b1 = _c(b1, np.float32)
    w2 = _c(w2, np.float32)
    dx = np.empty(x.shape, np.float64)
    dlogit = np.empty((R, k), np.float64)
    dW1 = np.empty((k, k), np.float64)
    db1 = np.empty(k, np.float64)
    dw2 = np.empty(k, np.float64)
    db2 = np.zeros(1, np.float64)
    st = _load().moce_oracle_backward(_p(x), _p(dy), N, H, W, C, _LAYOUT[layout], R, k, _p(pidx),
                                      _p(plog), _p(resid) if resid.size else None, int(resid.size),
                                      _p(W1), _p(b1), _p(w2), float(b2), float(tau_min),
                                      float(tau_max), _p(dx), _p(dlogit), _p(dW1), _p(db1),
                                      _p(dw2), _p(db2))
    if st != OK:
        raise OracleError(st, "backward")
    return {"dx": dx, "dlogit": dlogit, "dW1": dW1, "db1": db1, "dw2": dw2, "db2": float(db2[0])}


def pack(support_idx: np.ndarray, support_logits: np.ndarray, C: int):
    """Deployment packing: rows sorted by (logit desc, index asc), U ascending.

    Returns (packed_idx [R,k] int32, packed_logits [R,k] float32, resid int32[|U|]).
    """
    si = _c(support_idx, np.int32)
    sl = _c(support_logits, np.float32)
    R, k = si.shape
    pidx = np.empty((R, k), np.int32)
    plog = np.empty((R, k), np.float32)
    resid = np.empty(C, np.int32)
    nres = np.zeros(1, np.int32)
    st = _load().moce_oracle_pack(C, R, k, _p(si), _p(sl), _p(pidx), _p(plog), _p(resid), _p(nres))
    if st != OK:
        raise OracleError(st, "pack")
    return pidx, plog, resid[: int(nres[0])].copy()


def pool(x: np.ndarray, layout: str) -> np.ndarray:
    """Sec. 3.3: z = GAP(x), [N, C] float64."""
    x = _c(x, np.float32)
    if layout == "nhwc":
        N, H, W, C = x.shape
    else:
        N, C, H, W = x.shape
    z = np.empty((N, C), np.float64)
    _load().moce_oracle_pool(_p(x), N, H, W, C, _LAYOUT[layout], _p(z))
    return z


def gate(z: np.ndarray, packed_idx: np.ndarray, W1, b1, w2, b2: float, tau_min: float,
         tau_max: float, return_g: bool = False):
    """Eq. (tau): tau [N, R] float64 (and the pre-sigmoid gate values if asked)."""
    z = _c(z, np.float64)
    pidx = _c(packed_idx, np.int32)
    N, C = z.shape
    R, k = pidx.shape
    W1 = _c(W1, np.float32).reshape(k, k)
    b1 = _c(b1, np.float32).reshape(k)
    w2 = _c(w2, np.float32).reshape(k)
    tau = np.empty((N, R), np.float64)
    g = np.empty((N, R), np.float64)
    _load().moce_oracle_gate(_p(z), N, C, R, k, _p(pidx), _p(W1), _p(b1), _p(w2), float(b2),
                             float(tau_min), float(tau_max), _p(g), _p(tau))
    return (tau, g) if return_g else tau


def weights(tau: np.ndarray, packed_logits: np.ndarray) -> np.ndarray:
    """Eq. (weights): a [N, R, k] float64."""
    tau = _c(tau, np.float64)
    plog = _c(packed_logits, np.float32)
    N, R = tau.shape
    k = plog.shape[1]
    a = np.empty((N, R, k), np.float64)
    _load().moce_oracle_weights(_p(tau), N, R, k, _p(plog), _p(a))
    return a


def mix(x: np.ndarray, layout: str, packed_idx, a, resid) -> np.ndarray:
    """Eqs. (expert), (res): y with R + 1 channels in the layout of x, float64."""
    x = _c(x, np.float32)
    pidx = _c(packed_idx, np.int32)
    a = _c(a, np.float64)
    resid = _c(resid, np.int32)
    R, k = pidx.shape
    if layout == "nhwc":
        N, H, W, C = x.shape
        y = np.empty((N, H, W, R + 1), np.float64)
    else:
        N, C, H, W = x.shape
        y = np.empty((N, R + 1, H, W), np.float64)
    _load().moce_oracle_mix(_p(x), N, H, W, C, _LAYOUT[layout], R, k, _p(pidx), _p(a),
                            _p(resid) if resid.size else None, int(resid.size), _p(y))
    return y


def forward(x: np.ndarray, layout: str, packed_idx, packed_logits, resid, W1, b1, w2, b2,
            tau_min: float, tau_max: float, intermediates: bool = False):
    """The whole layer on packed supports. Returns y (float64), or (y, z, tau, a)."""
    x = _c(x, np.float32)
    pidx = _c(packed_idx, np.int32)
    plog = _c(packed_logits, np.float32)
    resid = _c(resid, np.int32)
    R, k = pidx.shape
    if layout == "nhwc":
        N, H, W, C = x.shape
        y = np.empty((N, H, W, R + 1), np.float64)
    else:
        N, C, H, W = x.shape
        y = np.empty((N, R + 1, H, W), np.float64)
    W1 = _c(W1, np.float32).reshape(k, k)
    b1 = _c(b1, np.float32).reshape(k)
    w2 = _c(w2, np.float32).reshape(k)
    z = np.empty((N, C), np.float64) if intermediates else None
    tau = np.empty((N, R), np.float64) if intermediates else None
    a = np.empty((N, R, k), np.float64) if intermediates else None
    st = _load().moce_oracle_forward(_p(x), N, H, W, C, _LAYOUT[layout], R, k, _p(pidx), _p(plog),
                                     _p(resid) if resid.size else None, int(resid.size), _p(W1),
                                     _p(b1), _p(w2), float(b2), float(tau_min), float(tau_max),
                                     _p(y), _p(z), _p(tau), _p(a))
    if st != OK:
        raise OracleError(st, "forward")
    return (y, z, tau, a) if intermediates else y


def bruteforce_forward(x: np.ndarray, layout: str, L: np.ndarray, k: int, W1, b1, w2, b2,
                       tau_min: float, tau_max: float) -> np.ndarray:
    """Independent dense restatement from the full routing matrix L [R, C] (tiny shapes only)."""
    x = _c(x, np.float32)
    L = _c(L, np.float32)
    R = L.shape[0]
    if layout == "nhwc":
        N, H, W, C = x.shape
        y = np.empty((N, H, W, R + 1), np.float64)
    else:
        N, C, H, W = x.shape
        y = np.empty((N, R + 1, H, W), np.float64)
    W1 = _c(W1, np.float32).reshape(k, k)
    b1 = _c(b1, np.float32).reshape(k)
    w2 = _c(w2, np.float32).reshape(k)
    st = _load().moce_oracle_bruteforce_forward(_p(x), N, H, W, C, _LAYOUT[layout], R, k, _p(L),
                                                _p(W1), _p(b1), _p(w2), float(b2), float(tau_min),
                                                float(tau_max), _p(y))
    if st != OK:
        raise OracleError(st, "bruteforce_forward")
    return y


class _use_library:
    """Temporarily route this module's calls to another build of the oracle.

    Used only by the mutation test, which compiles copies of the oracle with a
    planted mistake and checks that the pins reject each copy.
    """

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib
        self._saved = _load()
        _lib = None
        lib = ctypes.CDLL(self.path)
        # reuse the argtypes of the real build
        for name in ("moce_oracle_topk", "moce_oracle_pack", "moce_oracle_pool", "moce_oracle_gate",
                     "moce_oracle_weights", "moce_oracle_mix", "moce_oracle_forward",
                     "moce_oracle_bruteforce_forward", "moce_oracle_coverage",
                     "moce_oracle_backward"):
            src, dst = getattr(self._saved, name), getattr(lib, name)
            dst.argtypes, dst.restype = src.argtypes, src.restype
        _lib = lib
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self._saved
        return False


def dynamic_logits(x: np.ndarray, layout: str, L, Wh, bh, V, Q):
    """Eq. (dynamic): per-example logits L_e(X) = L_e + <q_e (.) h(z), v_c>, h(z) = ReLU(W_h z + b_h).

    L [R, C], Wh [d, C], bh [d], V [C, d], Q [R, d]. Returns (h [N, d], Ldyn [N, R, C]), float64.
    """
    x = _c(x, np.float32)
    if layout == "nhwc":
        N, H, W, C = x.shape
    else:
        N, C, H, W = x.shape
    L = _c(L, np.float32)
    R = L.shape[0]
    Wh = _c(Wh, np.float32)
    d = Wh.shape[0]
    h = np.empty((N, d), np.float64)
    Ld = np.empty((N, R, C), np.float64)
    st = _load().moce_oracle_dynamic_logits(_p(x), N, H, W, C, _LAYOUT[layout], R, d, _p(L), _p(Wh),
                                            _p(_c(bh, np.float32)), _p(_c(V, np.float32)),
                                            _p(_c(Q, np.float32)), _p(h), _p(Ld))
    if st != OK:
        raise OracleError(st, "dynamic_logits")
    return h, Ld


def dynamic_forward(x: np.ndarray, layout: str, L, Wh, bh, V, Q, k: int, W1, b1, w2, b2: float,
                    tau_min: float, tau_max: float):
    """The input-conditioned support variant (Sec. 5, Eq. dynamic), inference path.

    Per example: the logits of Eq. (dynamic); S_e(X) = TopK(L_e(X), k) decided on the float32
    values (the precision of the device path), in deployment order; U(X) the channels no
    expert of that example selects; the gate reads z at S_e(X) and the weights use the selected
    L_e(X) values (Eq. weights); then Eqs. (expert) and (res). Returns a dict: y, idx [N, R, k],
    logits [N, R, k] (float32), resid (a list of N int32 arrays), h [N, d], Ldyn [N, R, C].
    """
    h, Ld = dynamic_logits(x, layout, L, Wh, bh, V, Q)
    N, R, C = Ld.shape
    ys, idxs, lgs, resids = [], [], [], []
    for n in range(N):
        Lf = Ld[n].astype(np.float32)
        idx, lg = topk(Lf, k)
        pidx, plog, resid = pack(idx, lg, C)
        ys.append(forward(x[n:n + 1], layout, pidx, plog, resid, W1, b1, w2, b2, tau_min,
                          tau_max))
        idxs.append(pidx)
        lgs.append(plog)
        resids.append(resid)
    y = np.concatenate(ys, axis=0) if ys else np.zeros((0,), np.float64)
    return {"y": y, "idx": np.stack(idxs) if idxs else np.zeros((0, R, k), np.int32),
            "logits": np.stack(lgs) if lgs else np.zeros((0, R, k), np.float32),
            "resid": resids, "h": h, "Ldyn": Ld}
