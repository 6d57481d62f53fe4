"""Input-conditioned supports, Eq. (dynamic), on the GPU against the CPU oracle.

Selection is integer work decided on float32 logits. The device computes the
example's logits L_e(X) in fp32; the oracle computes them in double. The test
activations lie on a grid of 1/16, so every partial sum of the pool is exact
in fp32 and the device's z differs from the exact mean only by the rounding
of the final division. Each device logit then differs from the exact value by
at most tol[n,e,c], a worst-case bound of fp32 summation (any order: n terms
err by at most (n + 2) u times the sum of their magnitudes, u = 2^-24):
  z:    u |z|
  h_j:  dh_j = (ceil(C/32) + 10) u S_j, S_j = sum_c |W_h,jc z_c| + |b_h,j|
  L:    tol = 2 u |L_ec| + sum_j |q_ej v_cj| ((d + 4) u |h_j| + dh_j)
A row's selection is decided when every exact top-k value minus its bound
exceeds every other value plus its bound; there the device must select the
oracle's channels. Its order (the gate's positional input) is decided when
neighbouring exact values separate the same way; then it must match too.
Elsewhere the device's choice must be a possible top k (each selected value
plus its bound reaches the k-th largest lower bound) in an order the bounds
allow, and only outputs that depend on decided rows are compared.
"""
import numpy as np
import pytest

import oracle
from moce_cases import TOL, assert_close
from paper_2608_23794_gb300 import synth

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23794_gb300 import build
    build.build()


CFG = synth.CONFIGS
LC = synth.LayerConfig
CASES = {
    "tiny_f32_nchw": (CFG["tiny_f32_nchw"], 8),
    "ragged_bf16_nhwc": (LC("ragged_bf16_nhwc", 3, 9, 11, 72, 9, 5, "bf16", "nhwc", "relu", 60), 6),
    "odd_f32_nhwc": (LC("odd_f32_nhwc", 2, 5, 7, 60, 12, 6, "f32", "nhwc", "gelu", 50), 3),
    "rn50_stage1_reduce": (CFG["rn50_stage1_reduce"].replace(N=3), 32),
    "rn50_stage3_reduce": (CFG["rn50_stage3_reduce"].replace(N=2), 32),
    "vitb_ffn_exit_k32": (CFG["vitb_ffn_exit_k32"].replace(N=2), 32),
    "vitb_ffn_exit_k384": (CFG["vitb_ffn_exit_k384"].replace(N=1), 16),
    # degenerate shapes: every channel selected (U(X) empty), a rank-1 router, a channel count
    # that leaves a bitmap word partly unused, one example at one position
    "k_eq_c": (LC("k_eq_c", 2, 3, 4, 24, 5, 24, "f32", "nhwc", "relu", 24), 4),
    "d1_c70": (LC("d1_c70", 3, 5, 3, 70, 11, 6, "bf16", "nhwc", "gelu", 60), 1),
    "n1_hw1": (LC("n1_hw1", 1, 1, 1, 40, 9, 3, "f32", "nchw", "relu", 30), 2),
}


def _cu(a, dt=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dt)


def _setup(cfg, d, seed=5):
    from paper_2608_23794_gb300 import moce
    lay = synth.make_layer(cfg, seed=seed)
    xv, xb = synth.make_dynamic_x(cfg, seed=seed, grid=1.0 / 16)
    rt = synth.make_router(cfg, d, seed=seed)
    if xb is not None:
        x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    else:
        x = _cu(xv)
    router = moce.DynamicRouter(_cu(rt["L"]), _cu(rt["Wh"]), _cu(rt["bh"]), _cu(rt["V"]),
                                _cu(rt["Q"]))
    gate = (_cu(lay.W1), _cu(lay.b1), _cu(lay.w2), _cu(lay.b2))
    return lay, xv, x, rt, router, gate


U32 = 2.0 ** -24


def _tolerance(rt, h, z):
    """tol[n, e, c]: the bound of the module docstring."""
    L, Wh, bh, V, Q = (rt[k].astype(np.float64) for k in ("L", "Wh", "bh", "V", "Q"))
    C, d = Wh.shape[1], Wh.shape[0]
    S = np.abs(z) @ np.abs(Wh).T + np.abs(bh)                       # [N, d]
    dh = ((C + 31) // 32 + 10) * U32 * S                             # [N, d]
    hterm = (d + 4) * U32 * np.abs(h) + dh                            # [N, d]
    qv = np.abs(Q)[:, None, :] * np.abs(V)[None, :, :]                # [R, C, d]
    return 2 * U32 * np.abs(L)[None] + np.einsum("ecj,nj->nec", qv, hterm)


def _compare(cfg, d, seed=5):
    from paper_2608_23794_gb300 import moce
    lay, xv, x, rt, router, gate = _setup(cfg, d, seed)
    N, R, k, C = cfg.N, cfg.C_out, cfg.k, cfg.C_in
    sup = moce._empty_supports(N, R, k, C, "cuda")
    y = moce.moce_forward_dynamic(x, cfg.layout, router, k, *gate, cfg.tau_min, cfg.tau_max,
                                  supports=sup)
    torch.cuda.synchronize()
    ref = oracle.dynamic_forward(xv, cfg.layout, rt["L"], rt["Wh"], rt["bh"], rt["V"], rt["Q"], k,
                                 lay.W1, lay.b1, lay.w2, float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    z = oracle.pool(xv, cfg.layout)
    tol = _tolerance(rt, ref["h"], z)
    Ld = ref["Ldyn"]
    gidx = sup.sup_idx.cpu().numpy()
    glog = sup.sup_logits.cpu().numpy()
    gnu = sup.n_resid.cpu().numpy()
    set_ok = np.ones((N, R), bool)    # the selected set is decided (and matched)
    order_ok = np.ones((N, R), bool)  # the set and its order are decided (and matched)
    for n in range(N):
        for e in range(R):
            row, tr = Ld[n, e], tol[n, e]
            sel = gidx[n, e]
            assert len(set(sel.tolist())) == k and sel.min() >= 0 and sel.max() < C
            # the device's logits at its own selection are within the bound of the exact values
            assert np.all(np.abs(glog[n, e] - row[sel]) <= tr[sel]), (n, e)
            assert np.all(np.diff(glog[n, e]) <= 0), "supports not in deployment order"
            # consecutive entries of the device's order are consistent with the exact values
            assert np.all(row[sel[:-1]] + tr[sel[:-1]] >= row[sel[1:]] - tr[sel[1:]]), (n, e)
            top = ref["idx"][n, e]
            rest = np.setdiff1d(np.arange(C), top)
            lo = (row[top] - tr[top]).min()
            hi = (row[rest] + tr[rest]).max() if rest.size else -np.inf
            if lo > hi:
                assert set(sel.tolist()) == set(top.tolist()), (n, e)
                # the order (the gate's positional input) is decided where neighbours separate
                if np.all(row[top[:-1]] - tr[top[:-1]] > row[top[1:]] + tr[top[1:]]):
                    assert np.array_equal(sel, top), (n, e)
                else:
                    order_ok[n, e] = False
            else:
                set_ok[n, e] = order_ok[n, e] = False
                kth_lo = np.sort(row - tr)[::-1][k - 1]
                assert np.all(row[sel] + tr[sel] >= kth_lo), (n, e)
    yg = y.float().cpu().numpy().astype(np.float64)
    yr = ref["y"]
    xd = xv.astype(np.float64)
    ch = -1 if cfg.layout == "nhwc" else 0
    tol_y = TOL[cfg.dtype]
    for n in range(N):
        take = lambda a, idx: np.take(a[n], idx, axis=ch)
        decided = np.where(order_ok[n])[0]
        assert_close(take(yg, decided), take(yr, decided), cfg.dtype, f"routed y of example {n}")
        for e in np.where(~order_ok[n])[0]:
            # any valid order gives a convex mixture of the device's selected channels
            xs = take(xd, gidx[n, e])
            ye = take(yg, [e])
            lo_b, hi_b = xs.min(axis=ch, keepdims=True), xs.max(axis=ch, keepdims=True)
            slack = tol_y * (1 + np.maximum(np.abs(lo_b), np.abs(hi_b)))
            assert np.all(ye >= lo_b - slack) and np.all(ye <= hi_b + slack), (n, e)
        if set_ok[n].all():  # U(X) depends on the sets only
            assert gnu[n] == len(ref["resid"][n])
            assert_close(take(yg, [R]), take(yr, [R]), cfg.dtype, f"residual y of example {n}")
    return set_ok, order_ok


# fewest rows (of N C_out) whose set and order the bounds must decide, so that the exact
# comparison is exercised (large k leaves many near-equal neighbours in a support)
MIN_DECIDED = {"tiny_f32_nchw": 1.0, "ragged_bf16_nhwc": 1.0, "odd_f32_nhwc": 1.0,
               "k_eq_c": 0.5, "d1_c70": 0.9, "n1_hw1": 1.0,
               "rn50_stage1_reduce": 0.8, "rn50_stage3_reduce": 0.1, "vitb_ffn_exit_k32": 0.05,
               "vitb_ffn_exit_k384": 0.0}


@pytest.mark.parametrize("name", list(CASES))
def test_dynamic_matches_oracle(name):
    cfg, d = CASES[name]
    set_ok, order_ok = _compare(cfg, d)
    assert order_ok.mean() >= MIN_DECIDED[name]
    assert set_ok.mean() >= 0.5


def test_dynamic_supports_differ_between_examples():
    from paper_2608_23794_gb300 import moce
    cfg, d = CASES["rn50_stage1_reduce"]
    _, _, x, _, router, gate = _setup(cfg, d)
    sup = moce._empty_supports(cfg.N, cfg.C_out, cfg.k, cfg.C_in, "cuda")
    moce.moce_forward_dynamic(x, cfg.layout, router, cfg.k, *gate, cfg.tau_min, cfg.tau_max,
                              supports=sup)
    s = sup.sup_idx.cpu().numpy()
    assert not np.array_equal(s[0], s[1])


def test_dynamic_without_router_signal_is_the_static_layer():
    """q = 0: every example selects TopK(L); the supports equal the packed static ones bit for
    bit and y equals the static forward's."""
    from paper_2608_23794_gb300 import moce
    cfg, d = CASES["rn50_stage1_reduce"]
    lay, xv, x, rt, router, gate = _setup(cfg, d)
    router.Q.zero_()
    sup = moce._empty_supports(cfg.N, cfg.C_out, cfg.k, cfg.C_in, "cuda")
    yd = moce.moce_forward_dynamic(x, cfg.layout, router, cfg.k, *gate, cfg.tau_min, cfg.tau_max,
                                   supports=sup)
    pidx, plog, resid = oracle.pack(*oracle.topk(rt["L"], cfg.k), cfg.C_in)
    for n in range(cfg.N):
        assert np.array_equal(sup.sup_idx[n].cpu().numpy(), pidx)
        assert np.array_equal(sup.sup_logits[n].cpu().numpy().view(np.uint32), plog.view(np.uint32))
        assert int(sup.n_resid[n]) == len(resid)
    idx_t, lg_t = moce.moce_topk_supports(router.logits, cfg.k)
    packed = moce.moce_pack_supports(idx_t, lg_t, cfg.C_in)
    ys = moce.moce_forward(x, cfg.layout, packed, *gate, cfg.tau_min, cfg.tau_max)
    # two results of fp32 sums in different orders, each rounded to bf16: one ulp apart at most
    a = yd.float().cpu().numpy().astype(np.float64)
    b = ys.float().cpu().numpy().astype(np.float64)
    assert np.all(np.abs(a - b) <= 2.0 ** -7 * np.abs(b) + 1e-5)


def test_dynamic_stages_compose():
    """moce_pool + moce_dynamic_supports + moce_forward_supports == moce_forward_dynamic, bit for
    bit, and U(X) is the complement of the example's selections, ascending."""
    from paper_2608_23794_gb300 import moce
    cfg, d = CASES["ragged_bf16_nhwc"]
    _, _, x, _, router, gate = _setup(cfg, d)
    N, R, k, C = cfg.N, cfg.C_out, cfg.k, cfg.C_in
    y1 = moce.moce_forward_dynamic(x, cfg.layout, router, k, *gate, cfg.tau_min, cfg.tau_max)
    z = moce.moce_pool(x, cfg.layout)
    sup = moce.moce_dynamic_supports(z, router, k)
    y2 = moce.moce_forward_supports(x, cfg.layout, sup, *gate, cfg.tau_min, cfg.tau_max)
    assert torch.equal(y1, y2)
    idx = sup.sup_idx.cpu().numpy()
    res = sup.resid_idx.cpu().numpy()
    for n in range(N):
        want = np.setdiff1d(np.arange(C), idx[n].ravel())
        m = int(sup.n_resid[n])
        assert m == len(want) and np.array_equal(res[n, :m], want)


def test_mix_entry_point_matches_the_step_path():
    """moce_gate + moce_mix (shared supports) give the bytes of the step path's forward."""
    from paper_2608_23794_gb300 import moce
    from moce_cases import device_tensors
    cfg = CFG["rn50_stage3_reduce"].replace(N=2)
    lay = synth.make_layer(cfg, seed=2)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    ws = moce.Workspace(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k)
    y_steps = moce.moce_forward(dev["x"], cfg.layout, packed, dev["W1"], dev["b1"], dev["w2"],
                                dev["b2"], cfg.tau_min, cfg.tau_max, ws=ws, path="steps")
    z = moce.moce_pool(dev["x"], cfg.layout)
    tau, a = moce.moce_gate(z, packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"], cfg.tau_min,
                            cfg.tau_max)
    y_mix = moce.moce_mix(dev["x"], cfg.layout, packed.packed_idx.view(cfg.C_out, cfg.k), a,
                          packed.resid_idx, packed.n_resid, ws)
    assert torch.equal(y_steps, y_mix)


@pytest.mark.parametrize("dtype,layout,C", [("f32", "nchw", 40), ("f32", "nhwc", 40),
                                            ("bf16", "nhwc", 72), ("bf16", "nhwc", 512)])
def test_mix_holds_per_example_counts_to_the_row(dtype, layout, C):
    """A per-example |U| above C_in mixes the whole row of C_in entries; one below 0 mixes none.

    (Every mixing kernel: the NCHW one, the generic NHWC one, the tiled bf16 one and, from
    512 channels, the wide one.)
    """
    from paper_2608_23794_gb300 import moce
    N, H, W, R, k = 2, 5, 7, 9, 4
    rng = np.random.default_rng(7)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    shape = (N, C, H, W) if layout == "nchw" else (N, H, W, C)
    x = torch.from_numpy(rng.standard_normal(shape).astype(np.float32)).to("cuda", tdt)
    sidx = _cu(np.stack([rng.permutation(C)[: R * k].reshape(R, k) for _ in range(N)]), torch.int32)
    a = _cu(rng.random((N, R, k)).astype(np.float32))
    resid = _cu(np.stack([rng.permutation(C) for _ in range(N)]), torch.int32)
    ws = moce.Workspace(N, H, W, C, R, k)
    out = {}
    for name, counts in (("held", [C + 50, -3]), ("in_range", [C, 0])):
        out[name] = moce.moce_mix(x, layout, sidx, a, resid, _cu(np.array(counts), torch.int32), ws)
    torch.cuda.synchronize()
    assert torch.equal(out["held"], out["in_range"])
    yres = out["held"][..., R] if layout == "nhwc" else out["held"][:, R]
    assert torch.count_nonzero(yres[1]) == 0
    xm = x[0].float().mean(dim=-1 if layout == "nhwc" else 0)
    assert torch.allclose(yres[0].float(), xm, atol=1e-2 if dtype == "bf16" else 1e-5)
