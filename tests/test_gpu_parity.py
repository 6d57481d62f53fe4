"""CUDA path vs the CPU oracle, through the C ABI, on seeded synthetic layers.

Small cases are compared element by element at sizes that span several tiles
and a ragged tail; the five workload shapes at full size are compared on
whole sampled examples. Packing and index handling must be bit-exact."""
import numpy as np
import pytest

import oracle
from moce_cases import TOL, assert_close, device_tensors, gpu_forward, oracle_forward, oracle_packed
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

# reduced-N versions of every workload shape (full channel/expert/support sizes)
SMALL = {
    "tiny_f32_nchw": CFG["tiny_f32_nchw"],
    "rn50_stage1_reduce": CFG["rn50_stage1_reduce"].replace(N=3),
    "rn50_stage3_reduce": CFG["rn50_stage3_reduce"].replace(N=5),
    "rn50_stage4_reduce": CFG["rn50_stage4_reduce"].replace(N=5),
    "vitb_ffn_exit_k32": CFG["vitb_ffn_exit_k32"].replace(N=3),
    "vitb_ffn_exit_k96": CFG["vitb_ffn_exit_k96"].replace(N=2),
    "vitb_ffn_exit_k192": CFG["vitb_ffn_exit_k192"].replace(N=2),
    "vitb_ffn_exit_k384": CFG["vitb_ffn_exit_k384"].replace(N=2),
}


# ------------------------------------------------------------------ packing


@pytest.mark.parametrize("name", list(SMALL))
def test_pack_bit_exact(name):
    from paper_2608_23794_gb300 import moce
    lay = synth.make_layer(SMALL[name], seed=11)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], lay.cfg.C_in)
    pidx, plog, resid = oracle_packed(lay)
    assert packed.packed_idx.cpu().numpy().tobytes() == pidx.tobytes()
    assert packed.packed_logits.cpu().numpy().tobytes() == plog.tobytes()
    assert packed.n_resid == len(resid)
    assert packed.resid_idx[: packed.n_resid].cpu().numpy().tobytes() == resid.tobytes()


def test_pack_permutation_invariant_and_ties():
    from paper_2608_23794_gb300 import moce
    rng = np.random.default_rng(5)
    C, R, k = 300, 40, 24
    idx = np.stack([rng.choice(C, size=k, replace=False) for _ in range(R)]).astype(np.int32)
    lg = rng.standard_normal((R, k)).astype(np.float32)
    lg[:, 3] = lg[:, 7]
    lg[:, 5] = 0.0
    lg[:, 6] = -0.0
    ref = oracle.pack(idx, lg, C)
    for trial in range(3):
        perm = np.stack([rng.permutation(k) for _ in range(R)])
        pi = torch.from_numpy(np.take_along_axis(idx, perm, 1)).cuda()
        pl = torch.from_numpy(np.take_along_axis(lg, perm, 1)).cuda()
        p = moce.moce_pack_supports(pi, pl, C)
        assert p.packed_idx.cpu().numpy().tobytes() == ref[0].tobytes()
        assert p.packed_logits.cpu().numpy().tobytes() == ref[1].tobytes()
        assert p.resid_idx[: p.n_resid].cpu().numpy().tobytes() == ref[2].tobytes()


@pytest.mark.parametrize("bad", ["range_hi", "range_lo", "dup", "nan", "inf"])
def test_pack_rejects_bad_supports(bad):
    from paper_2608_23794_gb300 import moce
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
        lg[1, 0] = -np.inf
    with pytest.raises(moce.MoceError) as ei:
        moce.moce_pack_supports(torch.from_numpy(idx).cuda(), torch.from_numpy(lg).cuda(), 6)
    assert ei.value.status == moce.MOCE_ERR_BAD_SUPPORT


def test_pack_cyclic_supports_empty_and_full_residual():
    from paper_2608_23794_gb300 import moce
    for C, R, k in ((64, 16, 4), (64, 15, 4), (256, 10, 16)):
        idx = synth.cyclic_supports(C, R, k)
        lg = np.random.default_rng(0).standard_normal((R, k)).astype(np.float32)
        p = moce.moce_pack_supports(torch.from_numpy(idx).cuda(), torch.from_numpy(lg).cuda(), C)
        want = list(range(R * k, C)) if R * k < C else []
        assert p.resid_idx[: p.n_resid].cpu().tolist() == want


# ------------------------------------------------------------------ pool + gate


@pytest.mark.parametrize("name", list(SMALL))
def test_pool_and_gate(name):
    from paper_2608_23794_gb300 import moce
    cfg = SMALL[name]
    lay = synth.make_layer(cfg, seed=3)
    dev = device_tensors(lay)
    z = moce.moce_pool(dev["x"], cfg.layout).cpu().numpy()
    zref = oracle.pool(lay.x, cfg.layout)
    np.testing.assert_allclose(z, zref, rtol=1e-5, atol=1e-6)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    pidx, plog, _ = oracle_packed(lay)
    zt = torch.from_numpy(zref.astype(np.float32)).cuda()
    tau, a = moce.moce_gate(zt, packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"], cfg.tau_min,
                            cfg.tau_max)
    tref = oracle.gate(zref.astype(np.float32).astype(np.float64), pidx, lay.W1, lay.b1, lay.w2,
                       float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    np.testing.assert_allclose(tau.cpu().numpy(), tref, rtol=2e-5, atol=1e-6)
    aref = oracle.weights(tau.cpu().numpy().astype(np.float64), plog)
    np.testing.assert_allclose(a.cpu().numpy(), aref, rtol=2e-5, atol=1e-7)


GATE_BLOCKS = {
    # C_out not a multiple of the tiled gate's 64-expert block, k on its tiled path, C_in ragged
    "r70_k32": synth.LayerConfig("r70_k32", 3, 2, 2, 200, 70, 32, "bf16", "nhwc", "relu", 180),
    "r5_k64": synth.LayerConfig("r5_k64", 2, 2, 2, 300, 5, 64, "bf16", "nhwc", "gelu", 256),
    "r130_k128": synth.LayerConfig("r130_k128", 2, 2, 2, 256, 130, 128, "bf16", "nhwc", "relu", 224),
    "r100_k384": synth.LayerConfig("r100_k384", 1, 1, 1, 512, 100, 384, "bf16", "nhwc", "gelu", 448),
}


@pytest.mark.parametrize("name", list(GATE_BLOCKS))
def test_tiled_gate_partial_expert_blocks(name):
    """tau and the weights against the oracle when the last block of 64 experts is partial."""
    from paper_2608_23794_gb300 import moce
    cfg = GATE_BLOCKS[name]
    lay = synth.make_layer(cfg, seed=23)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    pidx, plog, _ = oracle_packed(lay)
    zref = oracle.pool(lay.x, cfg.layout)
    zt = torch.from_numpy(zref.astype(np.float32)).cuda()
    tau, a = moce.moce_gate(zt, packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"], cfg.tau_min,
                            cfg.tau_max)
    tref = oracle.gate(zref.astype(np.float32).astype(np.float64), pidx, lay.W1, lay.b1, lay.w2,
                       float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    np.testing.assert_allclose(tau.cpu().numpy(), tref, rtol=2e-5, atol=1e-6)
    aref = oracle.weights(tau.cpu().numpy().astype(np.float64), plog)
    np.testing.assert_allclose(a.cpu().numpy(), aref, rtol=2e-5, atol=1e-7)


POOL_SHAPES = {
    # (N, H, W, C, dtype, element offset of x): the tilings of the NHWC pool
    "many_spans_c256": (2, 56, 56, 256, "bf16", 0),
    "spans_capped_c2048": (3, 7, 7, 2048, "bf16", 0),
    "spans_c3072": (2, 14, 14, 3072, "bf16", 0),
    "five_spans_c1024": (70, 14, 14, 1024, "bf16", 0),
    "one_span_c1024": (160, 7, 7, 1024, "bf16", 0),
    "narrow_block_f32": (3, 5, 7, 60, "f32", 0),
    "narrow_block_bf16": (2, 9, 11, 72, "bf16", 0),
    "scalar_ragged_block": (2, 6, 6, 70, "bf16", 0),
    "unaligned_bf16": (2, 8, 8, 256, "bf16", 1),
    "unaligned_f32": (2, 8, 8, 128, "f32", 1),
    "one_position": (1, 1, 1, 8, "bf16", 0),
}


@pytest.mark.parametrize("name", list(POOL_SHAPES))
def test_pool_tilings(name):
    """z = GAP(x) against the oracle for one span and several per example, 16-byte and
    scalar loads, channel blocks narrower than 32 vectors and a ragged last block."""
    from paper_2608_23794_gb300 import moce
    N, H, W, C, dt, off = POOL_SHAPES[name]
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    rng = np.random.default_rng(17)
    xf = rng.standard_normal((N, H, W, C)).astype(np.float32)
    buf = torch.empty(N * H * W * C + off, dtype=tdt, device="cuda")
    x = buf[off:].view(N, H, W, C)
    x.copy_(torch.from_numpy(xf))
    z = moce.moce_pool(x, "nhwc").cpu().numpy()
    zref = oracle.pool(x.float().cpu().numpy(), "nhwc")
    np.testing.assert_allclose(z, zref, rtol=1e-5, atol=1e-6)


# ------------------------------------------------------------------ forward, element by element


@pytest.mark.parametrize("name", list(SMALL))
def test_forward_small(name):
    cfg = SMALL[name]
    lay = synth.make_layer(cfg, seed=1)
    y, packed, ws = gpu_forward(lay)
    yref, zref, tref, _ = oracle_forward(lay, intermediates=True)
    assert_close(y, yref, cfg.dtype)
    # the forward's own intermediates, read back from its workspace
    np.testing.assert_allclose(ws.z().cpu().numpy(), zref, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(ws.tau().cpu().numpy(), tref, rtol=2e-5, atol=1e-6)


EDGE = {
    # C % 64 != 0 (padded staging), odd R, odd k
    "c72_r9_k5": synth.LayerConfig("c72_r9_k5", 3, 9, 11, 72, 9, 5, "bf16", "nhwc", "relu", 60),
    # C % 8 != 0: scalar NHWC path
    "c100_r12_k7": synth.LayerConfig("c100_r12_k7", 2, 5, 7, 100, 12, 7, "bf16", "nhwc", "gelu", 90),
    # fp32 NHWC
    "f32_nhwc": synth.LayerConfig("f32_nhwc", 2, 6, 10, 128, 20, 8, "f32", "nhwc", "relu", 112),
    # bf16 NCHW
    "bf16_nchw": synth.LayerConfig("bf16_nchw", 2, 7, 9, 96, 16, 6, "bf16", "nchw", "gelu", 84),
    # k = 1: each expert copies one channel
    "k1": synth.LayerConfig("k1", 2, 8, 8, 64, 32, 1, "bf16", "nhwc", "relu", 56),
    # k = C_in: every expert reads every channel, U is empty
    "k_eq_c": synth.LayerConfig("k_eq_c", 2, 4, 4, 16, 4, 16, "bf16", "nhwc", "relu", 16),
    # a single position per example
    "hw1": synth.LayerConfig("hw1", 9, 1, 1, 256, 64, 16, "bf16", "nhwc", "relu", 224),
    # few experts (R smaller than the CTA's lane groups)
    "r3": synth.LayerConfig("r3", 2, 16, 16, 256, 3, 16, "bf16", "nhwc", "relu", 224),
    # large k with small C_out
    "k200_r5": synth.LayerConfig("k200_r5", 2, 5, 5, 512, 5, 200, "bf16", "nhwc", "relu", 448),
}


@pytest.mark.parametrize("name", list(EDGE))
def test_forward_edge_cases(name):
    cfg = EDGE[name]
    lay = synth.make_layer(cfg, seed=2)
    y, _, _ = gpu_forward(lay)
    assert_close(y, oracle_forward(lay), cfg.dtype)


def test_forward_empty_residual_is_zero():
    cfg = synth.LayerConfig("cyc", 2, 7, 7, 64, 16, 4, "bf16", "nhwc", "relu", 64)
    lay = synth.make_layer(cfg, seed=0)
    lay.support_idx = synth.cyclic_supports(64, 16, 4)
    y, packed, _ = gpu_forward(lay)
    assert packed.n_resid == 0
    assert np.all(y[..., 16] == 0.0)
    assert_close(y, oracle_forward(lay), "bf16")


def test_forward_layouts_and_dtypes_agree():
    base = synth.LayerConfig("lay", 2, 12, 12, 128, 24, 8, "f32", "nhwc", "relu", 112)
    lay = synth.make_layer(base, seed=4)
    y_nhwc, _, _ = gpu_forward(lay)
    lay_c = synth.make_layer(base.replace(layout="nchw"), seed=4)
    assert np.array_equal(lay_c.x, synth.x_to_layout(lay.x, "nhwc", "nchw"))
    y_nchw, _, _ = gpu_forward(lay_c)
    np.testing.assert_allclose(synth.x_to_layout(y_nhwc, "nhwc", "nchw"), y_nchw, rtol=1e-5,
                               atol=1e-6)


def test_forward_empty_batch():
    from paper_2608_23794_gb300 import moce
    cfg = synth.LayerConfig("e", 0, 4, 4, 64, 8, 4, "bf16", "nhwc", "relu", 56)
    lay = synth.make_layer(cfg.replace(N=1), seed=0)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], 64)
    x = dev["x"][:0]
    y = moce.moce_forward(x, "nhwc", packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"], 0.2, 6.0,
                          ws=moce.Workspace(1, 4, 4, 64, 8, 4))
    assert y.shape == (0, 4, 4, 9)


def test_forward_is_deterministic_and_reuses_workspace():
    cfg = SMALL["rn50_stage1_reduce"]
    lay = synth.make_layer(cfg, seed=8)
    dev = device_tensors(lay)
    y1, packed, ws = gpu_forward(lay, dev=dev)
    y2, _, _ = gpu_forward(lay, dev=dev, ws=ws)
    y3, _, _ = gpu_forward(lay, dev=dev, ws=ws)
    assert np.array_equal(y1, y2) and np.array_equal(y2, y3)


def test_temperature_limits_on_device():
    # tau fixed high -> support mean; tau fixed tiny -> the argmax-logit channel (Sec. 3.3)
    cfg = synth.LayerConfig("lim", 2, 8, 8, 128, 16, 8, "f32", "nhwc", "relu", 112)
    lay = synth.make_layer(cfg, seed=6)
    pidx, plog, _ = oracle_packed(lay)
    for T, check in ((1e4, "mean"), (1e-3, "argmax")):
        y, _, _ = gpu_forward(lay.__class__(**{**lay.__dict__, "cfg": cfg.replace(tau_min=T, tau_max=T)}))
        x = lay.x.astype(np.float64)
        for e in range(cfg.C_out):
            if check == "mean":
                np.testing.assert_allclose(y[..., e], x[..., pidx[e]].mean(-1), rtol=1e-3, atol=1e-4)
            elif plog[e, 0] - plog[e, 1] >= 0.05:
                np.testing.assert_allclose(y[..., e], x[..., pidx[e, 0]], rtol=1e-6, atol=1e-7)


# ------------------------------------------------------------------ full-size workloads, sampled


FULL = ["rn50_stage1_reduce", "rn50_stage3_reduce", "rn50_stage4_reduce", "vitb_ffn_exit_k32",
        "vitb_ffn_exit_k96", "vitb_ffn_exit_k192", "vitb_ffn_exit_k384"]


@pytest.mark.parametrize("name", FULL)
def test_forward_full_size_sampled(name):
    cfg = CFG[name]
    lay = synth.make_layer(cfg, seed=0)
    y, _, ws = gpu_forward(lay)
    ex = [0, cfg.N // 2, cfg.N - 1]
    yref = oracle_forward(lay, examples=ex)
    assert_close(y[ex], yref, cfg.dtype)
    # properties over the whole output: finite, residual channel present
    assert np.isfinite(y).all()
    z = ws.z().cpu().numpy()
    np.testing.assert_allclose(z[ex], oracle.pool(lay.x[ex], cfg.layout), rtol=1e-5, atol=1e-6)


# ------------------------------------------------------------------ every kernel path


PATHS = ["stream", "steps"]
PATH_CASES = {
    "rn50_stage1_reduce": SMALL["rn50_stage1_reduce"],
    "c72_r9_k5": EDGE["c72_r9_k5"],
    "k1": EDGE["k1"],
    "k_eq_c": EDGE["k_eq_c"],
    "hw1": EDGE["hw1"],
    "r3": EDGE["r3"],
    "f32_nhwc": EDGE["f32_nhwc"],
}


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("name", list(PATH_CASES))
def test_every_path_matches_oracle(name, path):
    from paper_2608_23794_gb300 import moce
    cfg = PATH_CASES[name]
    lay = synth.make_layer(cfg, seed=3)
    dev = device_tensors(lay)
    if moce.moce_forward_launches(dev["x"], cfg.layout, cfg.C_out, cfg.k, path=path) == 0:
        with pytest.raises(moce.MoceError):
            gpu_forward(lay, dev=dev, path=path)
        return
    y1, _, ws = gpu_forward(lay, dev=dev, path=path)
    assert_close(y1, oracle_forward(lay), cfg.dtype)
    # a second call on the same workspace gives the same bits
    y2, _, _ = gpu_forward(lay, dev=dev, ws=ws, path=path)
    assert np.array_equal(y1, y2)


@pytest.mark.parametrize("path", ["stream", "steps"])
def test_stage1_full_size_every_path(path):
    from paper_2608_23794_gb300 import moce
    cfg = CFG["rn50_stage1_reduce"]
    lay = synth.make_layer(cfg, seed=5)
    dev = device_tensors(lay)
    assert moce.moce_forward_launches(dev["x"], cfg.layout, cfg.C_out, cfg.k, path=path) >= 1
    y, _, _ = gpu_forward(lay, dev=dev, path=path)
    ex = [1, cfg.N // 3, cfg.N - 2]
    assert_close(y[ex], oracle_forward(lay, examples=ex), cfg.dtype)
    assert np.isfinite(y).all()
