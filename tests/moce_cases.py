"""Shared helpers for the GPU parity tests: move a synthetic layer to the
device, run the CUDA path through the binding, run the oracle on the same
inputs, and compare with the tolerances of the contract."""
from __future__ import annotations

import numpy as np

import oracle
from paper_2608_23794_gb300 import synth

# Contract tolerances: |y - y_ref| <= TOL + TOL*|y_ref| element-wise.
TOL = {"f32": 1e-5, "bf16": 2e-2}


def device_tensors(lay: synth.SyntheticLayer, device="cuda"):
    import torch
    cfg = lay.cfg
    if cfg.dtype == "bf16":
        x = torch.from_numpy(lay.x_bits.view(np.int16)).view(torch.bfloat16).to(device)
    else:
        x = torch.from_numpy(lay.x).to(device)
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).to(device=device, dtype=dt)
    return dict(
        x=x,
        support_idx=t(lay.support_idx, torch.int32),
        support_logits=t(lay.support_logits, torch.float32),
        W1=t(lay.W1, torch.float32),
        b1=t(lay.b1, torch.float32),
        w2=t(lay.w2, torch.float32),
        b2=t(lay.b2, torch.float32),
    )


def gpu_forward(lay: synth.SyntheticLayer, dev=None, ws=None, path="auto"):
    """Returns (y float64 numpy, packed, ws) from moce_pack_supports + moce_forward."""
    import torch
    from paper_2608_23794_gb300 import moce
    cfg = lay.cfg
    dev = dev or device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    if ws is None:
        ws = moce.Workspace(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k)
    y = moce.moce_forward(dev["x"], cfg.layout, packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"],
                          cfg.tau_min, cfg.tau_max, ws=ws, path=path)
    torch.cuda.synchronize()
    moce.moce_check_device_error(ws)
    return y.float().cpu().numpy().astype(np.float64), packed, ws


def oracle_packed(lay: synth.SyntheticLayer):
    return oracle.pack(lay.support_idx, lay.support_logits, lay.cfg.C_in)


def oracle_forward(lay: synth.SyntheticLayer, examples=None, intermediates=False):
    cfg = lay.cfg
    pidx, plog, resid = oracle_packed(lay)
    x = lay.x if examples is None else lay.x[np.asarray(examples)]
    return oracle.forward(x, cfg.layout, pidx, plog, resid, lay.W1, lay.b1, lay.w2,
                          float(lay.b2[0]), cfg.tau_min, cfg.tau_max, intermediates=intermediates)


def assert_close(got: np.ndarray, ref: np.ndarray, dtype: str, what: str = "y"):
    tol = TOL[dtype]
    err = np.abs(got - ref)
    bound = tol + tol * np.abs(ref)
    bad = err > bound
    if bad.any():
        i = np.unravel_index(np.argmax(err - bound), err.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} of {err.size} elements outside "
                             f"{tol} abs+rel; worst at {i}: got {got[i]!r} ref {ref[i]!r}")
    if dtype == "bf16":
        # Stronger than the contract: a correct fp32-accumulated result differs
        # from the exact value only by the final bf16 rounding (half an ulp,
        # at most 2^-8 relative) plus fp32 rounding far below that (the
        # absolute 1e-5 covers sums whose terms cancel).
        rb = np.abs(ref) * (2.0 ** -8) * (1 + 1e-3) + 1e-5
        badr = err > rb
        if badr.any():
            i = np.unravel_index(np.argmax(err - rb), err.shape)
            raise AssertionError(f"{what}: {int(badr.sum())} elements beyond the bf16 rounding "
                                 f"bound; worst at {i}: got {got[i]!r} ref {ref[i]!r}")
    return float(err.max()) if err.size else 0.0
