"""Pins of the CPU oracle to facts fixed by the paper and by mathematics.

None of these re-types the oracle's own formulas: each checks a worked
example, a closed form, an invariant the paper states, a special case that
reduces to a library routine, or a brute-force restatement on tiny inputs.
"""
import json
import math
import os

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

import oracle
from paper_2608_23794_gb300 import synth

GOLD_DIR = os.path.join(os.path.dirname(__file__), "golden")


def _rand_supports(rng, C, R, k):
    idx = np.stack([rng.choice(C, size=k, replace=False) for _ in range(R)]).astype(np.int32)
    lg = rng.standard_normal((R, k)).astype(np.float32)
    return idx, lg


# ---------------------------------------------------------------- worked example


def test_worked_tiny_layer():
    g = json.load(open(os.path.join(GOLD_DIR, "worked_tiny_layer.json")))
    x = np.array(g["x_nhwc"], np.float32)
    pidx, plog, resid = oracle.pack(np.array(g["support_idx"]), np.array(g["support_logits"]), g["C"])
    ex = g["expected"]
    assert pidx.tolist() == ex["packed_idx"]
    assert resid.tolist() == ex["resid"]
    y, z, tau, a = oracle.forward(x, "nhwc", pidx, plog, resid, np.array(g["W1"]), np.array(g["b1"]),
                                  np.array(g["w2"]), g["b2"], g["tau_min"], g["tau_max"],
                                  intermediates=True)
    tol = g["rel_tol"]
    np.testing.assert_allclose(z, ex["z"], rtol=tol)
    np.testing.assert_allclose(tau, ex["tau"], rtol=tol)
    np.testing.assert_allclose(a, ex["a"], rtol=tol)
    np.testing.assert_allclose(y, ex["y_nhwc"], rtol=tol)


# ---------------------------------------------------------------- packing


@pytest.mark.parametrize("seed", range(5))
def test_pack_equals_bruteforce_sort(seed):
    rng = np.random.default_rng(seed)
    C, R, k = 37, 9, 5
    idx, lg = _rand_supports(rng, C, R, k)
    lg[:, 1] = lg[:, 0]  # force ties in every row
    pidx, plog, resid = oracle.pack(idx, lg, C)
    for e in range(R):
        want = sorted(zip(idx[e].tolist(), lg[e].tolist()), key=lambda t: (-t[1], t[0]))
        assert pidx[e].tolist() == [t[0] for t in want]
        assert plog[e].tolist() == [t[1] for t in want]
    assert resid.tolist() == sorted(set(range(C)) - set(idx.ravel().tolist()))


def test_pack_permutation_invariant():
    rng = np.random.default_rng(3)
    C, R, k = 64, 12, 7
    idx, lg = _rand_supports(rng, C, R, k)
    ref = oracle.pack(idx, lg, C)
    for _ in range(4):
        perm = np.stack([rng.permutation(k) for _ in range(R)])
        got = oracle.pack(np.take_along_axis(idx, perm, 1), np.take_along_axis(lg, perm, 1), C)
        for a, b in zip(ref, got):
            assert a.tobytes() == b.tobytes()


def test_pack_ties_and_signed_zero():
    idx = np.array([[5, 2, 9, 0]], np.int32)
    lg = np.array([[0.0, -0.0, 1.5, 0.0]], np.float32)
    pidx, plog, _ = oracle.pack(idx, lg, 10)
    assert pidx.tolist() == [[9, 0, 2, 5]]


@pytest.mark.parametrize("bad", ["range_hi", "range_lo", "dup", "nan", "inf"])
def test_pack_rejects(bad):
    idx = np.array([[0, 1, 2], [3, 4, 5]], np.int32)
    lg = np.zeros((2, 3), np.float32)
    if bad == "range_hi":
        idx[1, 2] = 6
    elif bad == "range_lo":
        idx[0, 0] = -1
    elif bad == "dup":
        idx[1, 2] = 3
    elif bad == "nan":
        lg[0, 1] = np.nan
    else:
        lg[1, 0] = np.inf
    with pytest.raises(oracle.OracleError) as ei:
        oracle.pack(idx, lg, 6)
    assert ei.value.status == oracle.BAD_SUPPORT


@pytest.mark.parametrize("C,R,k", [(64, 16, 4), (64, 15, 4), (30, 4, 7), (256, 64, 16)])
def test_cyclic_supports_residual_closed_form(C, R, k):
    # Sec. 4.5 cyclic supports: experts cover channels 0 .. R*k-1 (mod C), so
    # U = {R*k, ..., C-1} when R*k < C and U is empty otherwise.
    idx = synth.cyclic_supports(C, R, k)
    lg = np.random.default_rng(0).standard_normal((R, k)).astype(np.float32)
    _, _, resid = oracle.pack(idx, lg, C)
    want = list(range(R * k, C)) if R * k < C else []
    assert resid.tolist() == want


def test_topk_equals_stable_argsort():
    rng = np.random.default_rng(11)
    L = rng.standard_normal((7, 40)).astype(np.float32)
    L[:, 5] = L[:, 6]  # ties
    idx, lg = oracle.topk(L, 9)
    ref = np.argsort(-L, axis=1, kind="stable")[:, :9]
    assert idx.tolist() == ref.tolist()
    assert lg.tolist() == np.take_along_axis(L, ref, 1).tolist()


# ---------------------------------------------------------------- coverage (Sec. 3.4)


def test_coverage_uniform_rows_are_zero():
    # equal logits in every row: p = 1/C, u = 1/C = ubar, so L_cov = 0 and dL_cov/dL = 0
    L = np.full((5, 12), 0.7, np.float32)
    loss, u, g = oracle.coverage(L, 1e-8)
    assert loss == 0.0
    np.testing.assert_allclose(u, 1.0 / 12, rtol=0, atol=1e-15)
    np.testing.assert_allclose(g, 0.0, atol=1e-12)


@pytest.mark.parametrize("a,b", [(0.0, 1.0), (2.5, -1.0), (-0.3, -0.3)])
def test_coverage_one_expert_two_channels_closed_form(a, b):
    # R = 1, C = 2: p = (s, 1 - s), s = 1 / (1 + exp(b - a)); ubar = 1/2, so
    # L_cov = 2 (s - 1/2)^2 / (1/4 + eps); dL_cov/da = 4 (s - 1/2) s (1 - s) / (1/4 + eps)
    eps = 1e-3
    s = 1.0 / (1.0 + math.exp(float(np.float32(b)) - float(np.float32(a))))
    loss, u, g = oracle.coverage(np.array([[a, b]], np.float32), eps)
    assert loss == pytest.approx(2 * (s - 0.5) ** 2 / (0.25 + eps), rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(u, [s, 1 - s], rtol=1e-12)
    da = 4 * (s - 0.5) * s * (1 - s) / (0.25 + eps)
    np.testing.assert_allclose(g[0], [da, -da], rtol=1e-9, atol=1e-15)


def test_coverage_row_shift_and_channel_permutation():
    rng = np.random.default_rng(4)
    L = rng.standard_normal((6, 9)).astype(np.float32)
    loss, _, g = oracle.coverage(L, 1e-6)
    # a constant added to one row leaves its softmax unchanged
    L2 = L.copy()
    L2[2] += np.float32(1.5)
    loss2, _, g2 = oracle.coverage(L2, 1e-6)
    assert loss2 == pytest.approx(loss, rel=1e-6)
    np.testing.assert_allclose(g2, g, rtol=1e-5, atol=1e-9)
    # permuting the channels of every row permutes u and the gradient
    perm = rng.permutation(9)
    loss3, _, g3 = oracle.coverage(L[:, perm], 1e-6)
    assert loss3 == pytest.approx(loss, rel=1e-12)
    np.testing.assert_allclose(g3, g[:, perm], rtol=1e-10, atol=1e-14)


def test_coverage_equals_numpy_definition_and_finite_differences():
    rng = np.random.default_rng(8)
    L = (1.7 * rng.standard_normal((4, 7))).astype(np.float32)
    eps = 1e-2
    loss, u, g = oracle.coverage(L, eps)
    # the definition with scipy's softmax over the channel axis
    P = sp_softmax(L.astype(np.float64), axis=1)
    uu = P.mean(axis=0)
    assert loss == pytest.approx(((uu - uu.mean()) ** 2).sum() / (uu.mean() ** 2 + eps), rel=1e-12)
    np.testing.assert_allclose(u, uu, rtol=1e-12)

    # central differences of the same definition in float64
    def f(Ld):
        Pd = sp_softmax(Ld, axis=1)
        ud = Pd.mean(axis=0)
        return ((ud - ud.mean()) ** 2).sum() / (ud.mean() ** 2 + eps)

    h = 1e-6
    fd = np.zeros_like(g)
    for e in range(L.shape[0]):
        for c in range(L.shape[1]):
            Lp, Lm = L.astype(np.float64), L.astype(np.float64)
            Lp[e, c] += h
            Lm[e, c] -= h
            fd[e, c] = (f(Lp) - f(Lm)) / (2 * h)
    np.testing.assert_allclose(g, fd, rtol=1e-6, atol=1e-10)
    assert abs(g.sum()) < 1e-12  # a common shift of all logits changes nothing


def test_coverage_rejects_non_finite():
    L = np.zeros((2, 3), np.float32)
    L[1, 2] = np.inf
    with pytest.raises(oracle.OracleError) as ei:
        oracle.coverage(L, 1e-8)
    assert ei.value.status == oracle.BAD_SUPPORT


# ---------------------------------------------------------------- pooling


@pytest.mark.parametrize("layout", ["nhwc", "nchw"])
def test_pool_closed_forms(layout):
    N, H, W, C = 2, 5, 3, 4
    const = np.full((N, H, W, C), 0.75, np.float32)
    ramp = np.broadcast_to(np.arange(H * W, dtype=np.float32).reshape(1, H, W, 1), (N, H, W, C))
    for x, want in ((const, 0.75), (ramp, (H * W - 1) / 2.0)):
        z = oracle.pool(synth.x_to_layout(np.ascontiguousarray(x), "nhwc", layout), layout)
        assert np.all(z == want)
    rnd = np.random.default_rng(0).standard_normal((N, H, W, C)).astype(np.float32)
    z = oracle.pool(synth.x_to_layout(rnd, "nhwc", layout), layout)
    np.testing.assert_allclose(z, rnd.astype(np.float64).mean(axis=(1, 2)), rtol=1e-12, atol=1e-15)


# ---------------------------------------------------------------- gate


def test_gate_zero_hidden_gives_sigmoid_of_bias():
    # W1 = 0, b1 = 0 -> h = 0 -> g = b2; sigma(0) = 1/2, sigma(ln 3) = 3/4.
    k, R, C = 3, 4, 10
    pidx = np.array([[0, 1, 2]] * R, np.int32)
    z = np.random.default_rng(1).standard_normal((2, C))
    zeros = np.zeros((k, k), np.float32)
    for b2, sig in ((0.0, 0.5), (math.log(3.0), 0.75)):
        tau = oracle.gate(z, pidx, zeros, np.zeros(k), np.ones(k), b2, 0.2, 6.0)
        np.testing.assert_allclose(tau, 0.2 + 5.8 * sig, rtol=1e-7)


def test_gate_reads_inputs_in_descending_logit_order_and_w1_rows_are_hidden_units():
    # W1 = E_01 (hidden unit 0 reads input position 1), w2 = e_0: g = ReLU(u_1),
    # the descriptor of each expert's SECOND most preferred channel.
    rng = np.random.default_rng(7)
    C, R, k = 12, 5, 3
    idx, lg = _rand_supports(rng, C, R, k)
    pidx, plog, _ = oracle.pack(idx, lg, C)
    z = rng.uniform(0.5, 2.0, size=(2, C))
    W1 = np.zeros((k, k), np.float32)
    W1[0, 1] = 1.0
    w2 = np.zeros(k, np.float32)
    w2[0] = 1.0
    _, g = oracle.gate(z, pidx, W1, np.zeros(k), w2, 0.0, 0.2, 6.0, return_g=True)
    for n in range(2):
        for e in range(R):
            second = idx[e][np.argsort(-lg[e], kind="stable")[1]]
            assert g[n, e] == pytest.approx(z[n, second], rel=1e-12)


def test_gate_relu_clamps():
    C, R, k = 4, 1, 2
    pidx = np.array([[0, 1]], np.int32)
    z = np.array([[-3.0, 2.0, 0.0, 0.0]])
    W1 = np.eye(2, dtype=np.float32)
    _, g = oracle.gate(z, pidx, W1, np.zeros(2), np.ones(2), 0.5, 0.2, 6.0, return_g=True)
    # h = ReLU([-3, 2]) = [0, 2]; g = 0 + 2 + 0.5
    assert g[0, 0] == pytest.approx(2.5, rel=1e-15)


def test_gate_range():
    cfg = synth.CONFIGS["tiny_f32_nchw"]
    lay = synth.make_layer(cfg, 5)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    z = oracle.pool(lay.x, cfg.layout) * 50.0
    tau = oracle.gate(z, pidx, lay.W1 * 10, lay.b1, lay.w2 * 10, float(lay.b2[0]), 0.2, 6.0)
    assert np.all(tau >= 0.2) and np.all(tau <= 6.0)


# ---------------------------------------------------------------- weights


def _weights_setup(seed=0, R=6, k=8):
    rng = np.random.default_rng(seed)
    idx, lg = _rand_supports(rng, 64, R, k)
    return oracle.pack(idx, lg, 64)


def test_weights_convex_and_order_invariant():
    pidx, plog, _ = _weights_setup()
    tau = np.random.default_rng(1).uniform(0.2, 6.0, size=(3, plog.shape[0]))
    a = oracle.weights(tau, plog)
    np.testing.assert_allclose(a.sum(-1), 1.0, rtol=1e-14)
    assert np.all(a > 0)
    # Sec. 3.3: along the temperature curve the ordering of the weights never changes;
    # positions are in descending-logit order, so a is non-increasing.
    assert np.all(np.diff(a, axis=-1) <= 1e-15)


def test_weights_unit_temperature_is_plain_softmax():
    pidx, plog, _ = _weights_setup(2)
    tau = np.ones((2, plog.shape[0]))
    a = oracle.weights(tau, plog)
    np.testing.assert_allclose(a[0], sp_softmax(plog.astype(np.float64), axis=-1), rtol=1e-13)


def test_weights_temperature_limits():
    pidx, plog, _ = _weights_setup(4)
    R, k = plog.shape
    a_hot = oracle.weights(np.full((1, R), 1e4), plog)
    spread = float(plog.max() - plog.min())
    assert np.max(np.abs(a_hot - 1.0 / k)) < 2 * spread / 1e4
    gaps = plog[:, 0] - plog[:, 1]
    a_cold = oracle.weights(np.full((1, R), 1e-3), plog)
    for e in range(R):
        if gaps[e] >= 0.05:
            assert a_cold[0, e, 0] == 1.0 and np.all(a_cold[0, e, 1:] < 1e-20)


# ---------------------------------------------------------------- mixing + residual


def test_mix_bounds_and_residual_mean():
    cfg = synth.CONFIGS["tiny_f32_nchw"]
    lay = synth.make_layer(cfg, 1)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    y = oracle.forward(lay.x, "nchw", pidx, plog, resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]),
                       0.2, 6.0)
    x = lay.x.astype(np.float64)
    for e in range(cfg.C_out):
        xs = x[:, pidx[e]]  # [N, k, H, W]
        assert np.all(y[:, e] >= xs.min(axis=1) - 1e-12)
        assert np.all(y[:, e] <= xs.max(axis=1) + 1e-12)
    assert len(resid) >= cfg.C_in - cfg.support_pool
    np.testing.assert_allclose(y[:, cfg.C_out], x[:, resid].mean(axis=1), rtol=1e-13)


def test_empty_residual_is_exactly_zero():
    C, R, k = 8, 4, 2  # cyclic supports cover all 8 channels
    idx = synth.cyclic_supports(C, R, k)
    lg = np.random.default_rng(0).standard_normal((R, k)).astype(np.float32)
    pidx, plog, resid = oracle.pack(idx, lg, C)
    assert resid.size == 0
    x = np.random.default_rng(1).uniform(1, 2, size=(2, 3, 3, C)).astype(np.float32)
    y = oracle.forward(x, "nhwc", pidx, plog, resid, np.zeros((k, k)), np.zeros(k), np.zeros(k),
                       0.0, 0.2, 6.0)
    assert np.all(y[..., R] == 0.0)


@pytest.mark.parametrize("layout", ["nhwc", "nchw"])
@pytest.mark.parametrize("seed", range(3))
def test_forward_equals_bruteforce(layout, seed):
    rng = np.random.default_rng(100 + seed)
    N, H, W, C, R, k = 2, 3, 4, 11, 5, 3
    L = rng.standard_normal((R, C)).astype(np.float32)
    L[:, 2] = L[:, 3]
    x = rng.standard_normal((N, H, W, C)).astype(np.float32)
    x = synth.x_to_layout(x, "nhwc", layout)
    W1 = rng.standard_normal((k, k)).astype(np.float32)
    b1 = rng.standard_normal(k).astype(np.float32)
    w2 = rng.standard_normal(k).astype(np.float32)
    b2 = float(rng.standard_normal())
    sidx, slog = oracle.topk(L, k)
    perm = np.stack([rng.permutation(k) for _ in range(R)])
    pidx, plog, resid = oracle.pack(np.take_along_axis(sidx, perm, 1),
                                    np.take_along_axis(slog, perm, 1), C)
    y = oracle.forward(x, layout, pidx, plog, resid, W1, b1, w2, b2, 0.2, 6.0)
    yb = oracle.bruteforce_forward(x, layout, L, k, W1, b1, w2, b2, 0.2, 6.0)
    np.testing.assert_allclose(y, yb, rtol=1e-12, atol=1e-13)


def test_fixed_temperature_is_a_linear_map():
    # tau_min = tau_max = T: the layer is y = W_eff x with W_eff built from
    # scipy's softmax of L/T on the support and 1/|U| on U; applied with einsum.
    rng = np.random.default_rng(9)
    N, H, W, C, R, k, T = 2, 4, 5, 16, 6, 4, 0.7
    idx, lg = _rand_supports(rng, 12, R, k)  # channels 12..15 stay in U
    x = rng.standard_normal((N, H, W, C)).astype(np.float32)
    pidx, plog, resid = oracle.pack(idx, lg, C)
    y = oracle.forward(x, "nhwc", pidx, plog, resid, rng.standard_normal((k, k)),
                       rng.standard_normal(k), rng.standard_normal(k), 0.3, T, T)
    Weff = np.zeros((R + 1, C))
    for e in range(R):
        Weff[e, idx[e]] = sp_softmax(lg[e].astype(np.float64) / T)
    Weff[R, resid] = 1.0 / len(resid)
    ref = np.einsum("oc,nhwc->nhwo", Weff, x.astype(np.float64))
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-13)


def test_layouts_agree():
    cfg = synth.CONFIGS["tiny_f32_nchw"]
    lay = synth.make_layer(cfg, 2)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    args = (pidx, plog, resid, lay.W1, lay.b1, lay.w2, float(lay.b2[0]), 0.2, 6.0)
    y_nchw = oracle.forward(lay.x, "nchw", *args)
    y_nhwc = oracle.forward(synth.x_to_layout(lay.x, "nchw", "nhwc"), "nhwc", *args)
    assert np.array_equal(synth.x_to_layout(y_nhwc, "nhwc", "nchw"), y_nchw)


# ---------------------------------------------------------------- backward (Sec. 3.2)


def _bwd_layer(layout, seed=0, N=2, H=3, W=4, C=12, R=5, k=3):
    rng = np.random.default_rng(seed)
    shape = (N, H, W, C) if layout == "nhwc" else (N, C, H, W)
    x = rng.standard_normal(shape).astype(np.float32)
    idx = np.stack([rng.permutation(C - 2)[:k] for _ in range(R)]).astype(np.int32)  # |U| >= 2
    lg = rng.standard_normal((R, k)).astype(np.float32)
    pidx, plog, resid = oracle.pack(idx, lg, C)
    W1 = (rng.standard_normal((k, k)) / np.sqrt(k)).astype(np.float32)
    b1 = (0.3 * rng.standard_normal(k)).astype(np.float32)
    w2 = rng.standard_normal(k).astype(np.float32)
    b2 = np.float32(0.2)
    yshape = (N, H, W, R + 1) if layout == "nhwc" else (N, R + 1, H, W)
    dy = rng.standard_normal(yshape).astype(np.float32)
    return x, pidx, plog, resid, W1, b1, w2, b2, dy


def _J(layout, x, pidx, plog, resid, W1, b1, w2, b2, dy, tmin=0.2, tmax=6.0):
    y = oracle.forward(x, layout, pidx, plog, resid, W1, b1, w2, float(b2), tmin, tmax)
    return float((y * dy.astype(np.float64)).sum())


@pytest.mark.parametrize("layout", ["nhwc", "nchw"])
def test_backward_equals_central_differences(layout):
    x, pidx, plog, resid, W1, b1, w2, b2, dy = _bwd_layer(layout, seed=3)
    g = oracle.backward(x, dy, layout, pidx, plog, resid, W1, b1, w2, float(b2), 0.2, 6.0)
    args = dict(x=x, pidx=pidx, plog=plog, resid=resid, W1=W1, b1=b1, w2=w2, b2=np.array([b2]),
                dy=dy)
    h = 2.0 ** -12  # exact in float32 for these magnitudes

    def fd(name, flat_i):
        a = {kk: (v.copy() if isinstance(v, np.ndarray) else v) for kk, v in args.items()}
        arr = a[name].reshape(-1)
        v0 = float(arr[flat_i])
        arr[flat_i] = np.float32(v0 + h)
        dp = float(arr[flat_i]) - v0
        jp = _J(layout, a["x"], a["pidx"], a["plog"], a["resid"], a["W1"], a["b1"], a["w2"],
                a["b2"][0], a["dy"])
        arr[flat_i] = np.float32(v0 - h)
        dm = v0 - float(arr[flat_i])
        jm = _J(layout, a["x"], a["pidx"], a["plog"], a["resid"], a["W1"], a["b1"], a["w2"],
                a["b2"][0], a["dy"])
        return (jp - jm) / (dp + dm)

    for name, got in [("x", g["dx"]), ("plog", g["dlogit"]), ("W1", g["dW1"]), ("b1", g["db1"]),
                      ("w2", g["dw2"]), ("b2", np.array([g["db2"]]))]:
        flat = got.reshape(-1)
        want = np.array([fd(name, i) for i in range(flat.size)])
        np.testing.assert_allclose(flat, want, rtol=1e-5, atol=1e-7, err_msg=name)


def test_backward_constant_temperature_is_the_transposed_linear_map():
    # tau_min = tau_max: tau does not depend on x or the gate, so the gate
    # gradients vanish, dx = W_eff^T dy with W_eff the per-example dense map of
    # Eq. (expert) and Eq. (res), and dlogit follows softmax(L / T) alone
    x, pidx, plog, resid, W1, b1, w2, b2, dy = _bwd_layer("nhwc", seed=5)
    T = 0.7
    g = oracle.backward(x, dy, "nhwc", pidx, plog, resid, W1, b1, w2, float(b2), T, T)
    for name in ("dW1", "db1", "dw2"):
        assert np.all(g[name] == 0.0), name
    assert g["db2"] == 0.0
    R, k = pidx.shape
    C = x.shape[-1]
    A = sp_softmax(plog.astype(np.float64) / T, axis=1)
    Weff = np.zeros((R + 1, C))
    for e in range(R):
        for i in range(k):
            Weff[e, pidx[e, i]] += A[e, i]
    if len(resid):
        Weff[R, resid] = 1.0 / len(resid)
    np.testing.assert_allclose(g["dx"], np.einsum("nhwe,ec->nhwc", dy.astype(np.float64), Weff),
                               rtol=1e-12, atol=1e-12)
    # dJ/dL_{e,i} = (1/T) a_i (da_i - sum_j a_j da_j), da_{e,i} = sum dy_e x_{S_e[i]}
    da = np.einsum("nhwe,nhwei->ei", dy.astype(np.float64)[..., :R],
                   x.astype(np.float64)[..., pidx])
    want = A * (da - (A * da).sum(1, keepdims=True)) / T
    np.testing.assert_allclose(g["dlogit"], want, rtol=1e-10, atol=1e-12)


def test_backward_is_linear_in_dy():
    x, pidx, plog, resid, W1, b1, w2, b2, dy = _bwd_layer("nhwc", seed=9)
    dy2 = np.random.default_rng(1).standard_normal(dy.shape).astype(np.float32)
    g1 = oracle.backward(x, dy, "nhwc", pidx, plog, resid, W1, b1, w2, float(b2), 0.2, 6.0)
    g2 = oracle.backward(x, dy2, "nhwc", pidx, plog, resid, W1, b1, w2, float(b2), 0.2, 6.0)
    g3 = oracle.backward(x, (dy + dy2).astype(np.float32), "nhwc", pidx, plog, resid, W1, b1, w2,
                         float(b2), 0.2, 6.0)
    # (dy + dy2 is rounded to float32: agreement to that rounding, relative to each array's scale)
    for name in ("dx", "dlogit", "dW1", "db1", "dw2"):
        want = g1[name] + g2[name]
        np.testing.assert_allclose(g3[name], want, rtol=0, atol=1e-6 * np.abs(want).max())


# ---------------------------------------------------------------- input-conditioned supports
# Eq. (dynamic): L_e(X)_c = L_{e,c} + <q_e (.) h(z), v_c>, h(z) = ReLU(W_h z + b_h).


def _dyn_setup(seed=0, N=2, H=3, W=5, C=20, R=6, d=4, layout="nhwc"):
    rng = np.random.default_rng(seed)
    shape = (N, H, W, C) if layout == "nhwc" else (N, C, H, W)
    x = rng.standard_normal(shape).astype(np.float32)
    L = rng.standard_normal((R, C)).astype(np.float32)
    Wh = (rng.standard_normal((d, C)) / np.sqrt(C)).astype(np.float32)
    bh = (0.5 + 0.1 * rng.standard_normal(d)).astype(np.float32)
    V = rng.standard_normal((C, d)).astype(np.float32)
    Q = rng.standard_normal((R, d)).astype(np.float32)
    return x, L, Wh, bh, V, Q


@pytest.mark.parametrize("zero", ["Q", "V", "h"])
def test_dynamic_offset_vanishes(zero):
    """No router signal (q = 0, v = 0, or h = ReLU(negative) = 0): L(X) is the static L exactly."""
    x, L, Wh, bh, V, Q = _dyn_setup(1)
    if zero == "Q":
        Q[:] = 0
    elif zero == "V":
        V[:] = 0
    else:
        Wh[:] = 0
        bh[:] = -1.0
    h, Ld = oracle.dynamic_logits(x, "nhwc", L, Wh, bh, V, Q)
    for n in range(x.shape[0]):
        assert np.array_equal(Ld[n], L.astype(np.float64))
    if zero == "h":
        assert np.all(h == 0.0)


def test_dynamic_single_coupling_lands_on_one_expert_and_channel():
    """One router unit j0 active (h = b at j0 only), q_e nonzero only at (e0, j0), v_c only at
    (c0, j0): the offset is q * b * v at exactly (e0, c0)."""
    x, L, Wh, bh, V, Q = _dyn_setup(2, d=3)
    Wh[:] = 0
    bh[:] = [0.0, 1.5, 0.0]
    Q[:] = 0
    V[:] = 0
    e0, c0 = 4, 13
    Q[e0, 1] = -2.0
    V[c0, 1] = 0.75
    Q[1, 0] = 9.0  # couples through unit 0, which is inactive
    V[3, 2] = 9.0  # unit 2 is inactive too
    h, Ld = oracle.dynamic_logits(x, "nhwc", L, Wh, bh, V, Q)
    want = L.astype(np.float64).copy()
    want[e0, c0] += -2.0 * 1.5 * 0.75
    for n in range(x.shape[0]):
        np.testing.assert_array_equal(Ld[n], want)
        np.testing.assert_array_equal(h[n], [0.0, 1.5, 0.0])


@pytest.mark.parametrize("layout", ["nhwc", "nchw"])
def test_dynamic_router_reads_the_pooled_descriptor(layout):
    """x constant over positions (x[n,p,c] = s_{n,c}) gives z = s; a router row that reads one
    channel c1 gives h_j = ReLU(w s_{c1} + b_j) for W_h [d][C] with row j = unit j."""
    N, H, W, C, R, d = 3, 2, 3, 10, 4, 2
    rng = np.random.default_rng(3)
    s = rng.standard_normal((N, C)).astype(np.float32)
    x = np.broadcast_to(s[:, None, None, :], (N, H, W, C)).astype(np.float32)
    if layout == "nchw":
        x = np.ascontiguousarray(x.transpose(0, 3, 1, 2))
    L = np.zeros((R, C), np.float32)
    Wh = np.zeros((d, C), np.float32)
    Wh[1, 7] = 2.0            # unit 1 reads channel 7
    bh = np.array([-5.0, 0.25], np.float32)
    V = np.zeros((C, d), np.float32)
    V[:, 1] = np.arange(C, dtype=np.float32)
    Q = np.zeros((R, d), np.float32)
    Q[:, 1] = 1.0
    h, Ld = oracle.dynamic_logits(x, layout, L, Wh, bh, V, Q)
    for n in range(N):
        hv = max(0.0, 2.0 * float(s[n, 7]) + 0.25)
        np.testing.assert_allclose(h[n], [0.0, hv], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(Ld[n], np.tile(hv * np.arange(C), (R, 1)), rtol=1e-12,
                                   atol=1e-12)


def test_dynamic_offset_has_rank_at_most_d_and_is_bilinear():
    x, L, Wh, bh, V, Q = _dyn_setup(4, C=24, R=10, d=3)
    _, Ld = oracle.dynamic_logits(x, "nhwc", L, Wh, bh, V, Q)
    for n in range(x.shape[0]):
        sv = np.linalg.svd(Ld[n] - L, compute_uv=False)
        assert sv[3] <= 1e-9 * sv[0]
    # powers of two keep the scaled float32 parameters exact
    _, Ld2 = oracle.dynamic_logits(x, "nhwc", L, Wh, bh, 2.0 * V, 4.0 * Q)
    np.testing.assert_allclose(Ld2 - L, 8.0 * (Ld - L), rtol=1e-12, atol=1e-12)


def test_dynamic_forward_without_router_signal_is_the_static_layer():
    """q = 0: every example selects TopK(L) and the layer is the static forward (Sec. 5: the
    variant replaces only the support of Eq. support)."""
    x, L, Wh, bh, V, Q = _dyn_setup(5, N=3, C=16, R=5)
    Q[:] = 0
    k = 4
    rng = np.random.default_rng(6)
    W1 = (rng.standard_normal((k, k)) / 2).astype(np.float32)
    b1 = rng.standard_normal(k).astype(np.float32)
    w2 = rng.standard_normal(k).astype(np.float32)
    out = oracle.dynamic_forward(x, "nhwc", L, Wh, bh, V, Q, k, W1, b1, w2, 0.3, 0.2, 6.0)
    pidx, plog, resid = oracle.pack(*oracle.topk(L, k), 16)
    ys = oracle.forward(x, "nhwc", pidx, plog, resid, W1, b1, w2, 0.3, 0.2, 6.0)
    np.testing.assert_array_equal(out["y"], ys)
    for n in range(3):
        assert np.array_equal(out["idx"][n], pidx) and np.array_equal(out["resid"][n], resid)


def test_dynamic_supports_follow_each_example():
    """A strong router term moves each example's supports toward the channels its own
    descriptor favours; U(X) is the complement of that example's union of supports."""
    N, H, W, C, R, d, k = 2, 2, 2, 12, 3, 1, 2
    x = np.zeros((N, H, W, C), np.float32)
    x[0, :, :, 0] = 1.0       # example 0 pools to channel 0 only
    x[1, :, :, 1] = 1.0       # example 1 pools to channel 1 only
    L = np.zeros((R, C), np.float32)
    L[:, 2:] = -np.arange(1, C - 1, dtype=np.float32) * 0.01  # static order: 0, 1 tie, then 2, 3, ...
    Wh = np.zeros((d, C), np.float32)
    Wh[0, 0] = 1.0            # h = ReLU(z_0): 1 for example 0, 0 for example 1
    bh = np.zeros(d, np.float32)
    V = np.zeros((C, d), np.float32)
    V[5, 0] = 10.0
    V[6, 0] = 9.0             # router pulls channels 5 and 6 up for example 0
    Q = np.ones((R, d), np.float32)
    W1 = np.zeros((k, k), np.float32)
    b1 = np.zeros(k, np.float32)
    w2 = np.zeros(k, np.float32)
    out = oracle.dynamic_forward(x, "nhwc", L, Wh, bh, V, Q, k, W1, b1, w2, 0.0, 1.0, 1.0)
    assert out["idx"][0].tolist() == [[5, 6]] * R
    assert out["idx"][1].tolist() == [[0, 1]] * R
    assert out["resid"][0].tolist() == [c for c in range(C) if c not in (5, 6)]
    assert out["resid"][1].tolist() == list(range(2, C))
    # tau = 1 (tau_min = tau_max): a = softmax of the example's selected logits
    a0 = sp_softmax(np.array([10.0, 9.0]) + L[0, [5, 6]])
    np.testing.assert_allclose(out["y"][0, 0, 0, 0], 0.0, atol=0)  # x is 0 on channels 5 and 6
    np.testing.assert_allclose(out["y"][1, 0, 0, :R], np.full(R, sp_softmax([0.0, 0.0])[1]),
                               rtol=1e-12)
    assert a0[0] > a0[1]
