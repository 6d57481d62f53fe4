"""Backward of the layer with static supports (Sec. 3.2) on the GPU against
the CPU oracle, through the C ABI.

Tolerance. The CUDA path sums in fp32 and the oracle in double on the same
inputs (bf16 inputs are exact in both). The longest fp32 sums are da over H W
positions and the parameter gradients over N C_out rows; their rounding error
is a few units of 2^-24 times the sum of the magnitudes of the terms, which
for these random inputs stays below 1e-4 of the largest gradient of each
output. Each gradient is therefore checked element-wise against
|got - ref| <= 1e-4 |ref| + 1e-4 max|ref|, with max|ref| the largest
magnitude of that output (sums with cancelling terms get the absolute part).
"""
import numpy as np
import pytest

import oracle
from moce_cases import device_tensors, oracle_packed
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
    # name: config (small cases span several tiles and a ragged tail)
    "tiny_f32_nchw": CFG["tiny_f32_nchw"],
    "ragged_f32_nhwc": LC("ragged_f32_nhwc", 3, 9, 11, 72, 9, 5, "f32", "nhwc", "relu", 60),
    "ragged_bf16_nchw": LC("ragged_bf16_nchw", 2, 13, 7, 48, 20, 40, "bf16", "nchw", "gelu", 48),
    # NHWC bf16 tiles: a ragged last tile, and C % 8 != 0 (no 16-byte channel groups)
    "ragged_bf16_nhwc": LC("ragged_bf16_nhwc", 3, 9, 11, 72, 9, 5, "bf16", "nhwc", "relu", 60),
    "odd_c_bf16_nhwc": LC("odd_c_bf16_nhwc", 2, 7, 5, 60, 12, 6, "bf16", "nhwc", "gelu", 50),
    "many_tiles_bf16_nhwc": LC("many_tiles_bf16_nhwc", 2, 23, 29, 128, 33, 12, "bf16", "nhwc",
                               "relu", 100),
    "k1": LC("k1", 2, 5, 5, 16, 16, 1, "f32", "nhwc", "relu", 16),
    "one_position": LC("one_position", 4, 1, 1, 40, 12, 7, "f32", "nhwc", "gelu", 30),
    "rn50_stage1_reduce": CFG["rn50_stage1_reduce"].replace(N=2),
    "rn50_stage3_reduce": CFG["rn50_stage3_reduce"].replace(N=3),
    "rn50_stage4_reduce": CFG["rn50_stage4_reduce"].replace(N=2),
    "vitb_ffn_exit_k32": CFG["vitb_ffn_exit_k32"].replace(N=2),
    "vitb_ffn_exit_k384": CFG["vitb_ffn_exit_k384"].replace(N=1),
}
RTOL = 1e-4


def _close(got, ref, what):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, what
    scale = float(np.abs(ref).max()) if ref.size else 0.0
    bound = RTOL * np.abs(ref) + RTOL * scale + 1e-30
    err = np.abs(got - ref)
    bad = err > bound
    if bad.any():
        i = np.unravel_index(np.argmax(err - bound), err.shape)
        raise AssertionError(f"{what}: {int(bad.sum())} of {err.size} outside; worst at {i}: "
                             f"got {got[i]!r} ref {ref[i]!r} (max|ref| {scale:.3g})")


def _run(cfg, seed=3):
    from paper_2608_23794_gb300 import moce
    lay = synth.make_layer(cfg, seed=seed)
    dyv, dyb = synth.make_dy(cfg, seed=seed)
    dev = device_tensors(lay)
    if dyb is not None:
        dy = torch.from_numpy(dyb.view(np.int16)).view(torch.bfloat16).cuda()
    else:
        dy = torch.from_numpy(dyv).cuda()
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    g = moce.moce_backward(dev["x"], dy, cfg.layout, packed, dev["W1"], dev["b1"], dev["w2"],
                           dev["b2"], cfg.tau_min, cfg.tau_max)
    torch.cuda.synchronize()
    pidx, plog, resid = oracle_packed(lay)
    ref = oracle.backward(lay.x, dyv, cfg.layout, pidx, plog, resid, lay.W1, lay.b1, lay.w2,
                          float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    return g, ref, (lay, dev, dy, packed)


@pytest.mark.parametrize("name", list(CASES))
def test_backward_matches_oracle(name):
    g, ref, _ = _run(CASES[name])
    _close(g.dx.cpu().numpy(), ref["dx"], "dx")
    _close(g.dlogits.cpu().numpy(), ref["dlogit"], "dlogits")
    _close(g.dW1.cpu().numpy(), ref["dW1"], "dW1")
    _close(g.db1.cpu().numpy(), ref["db1"], "db1")
    _close(g.dw2.cpu().numpy(), ref["dw2"], "dw2")
    _close(g.db2.cpu().numpy(), np.array([ref["db2"]]), "db2")


@pytest.mark.parametrize("name", ["rn50_stage1_reduce", "rn50_stage4_reduce"])
def test_backward_full_size_sampled(name):
    """The whole workload in the bench's launch configuration. dx of an example depends on that
    example alone, so sampled examples are compared with the oracle run on the example by itself;
    the parameter gradients are sums over examples, so the whole batch must give the sum of its
    two halves' gradients."""
    from paper_2608_23794_gb300 import moce
    cfg = CFG[name]
    lay = synth.make_layer(cfg, seed=5)
    dyv, dyb = synth.make_dy(cfg, seed=5)
    dev = device_tensors(lay)
    dy = torch.from_numpy(dyb.view(np.int16)).view(torch.bfloat16).cuda()
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    params = (dev["W1"], dev["b1"], dev["w2"], dev["b2"], cfg.tau_min, cfg.tau_max)
    g = moce.moce_backward(dev["x"], dy, cfg.layout, packed, *params)
    h = cfg.N // 2
    halves = [moce.moce_backward(dev["x"][a:b].contiguous(), dy[a:b].contiguous(), cfg.layout,
                                 packed, *params) for a, b in ((0, h), (h, cfg.N))]
    torch.cuda.synchronize()
    pidx, plog, resid = oracle_packed(lay)
    for n in (0, h + 1, cfg.N - 1):
        ref = oracle.backward(lay.x[n:n + 1], dyv[n:n + 1], cfg.layout, pidx, plog, resid, lay.W1,
                              lay.b1, lay.w2, float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
        _close(g.dx[n:n + 1].cpu().numpy(), ref["dx"], f"dx of example {n}")
    for f in ("dlogits", "dW1", "db1", "dw2", "db2"):
        whole = getattr(g, f).double().cpu().numpy()
        parts = sum(getattr(q, f).double().cpu().numpy() for q in halves)
        _close(whole, parts, f"{f}: whole batch against the sum of its halves")


def test_backward_is_deterministic():
    from paper_2608_23794_gb300 import moce
    g1, _, (lay, dev, dy, packed) = _run(CASES["rn50_stage3_reduce"])
    cfg = lay.cfg
    g2 = moce.moce_backward(dev["x"], dy, cfg.layout, packed, dev["W1"], dev["b1"], dev["w2"],
                            dev["b2"], cfg.tau_min, cfg.tau_max)
    for f in ("dx", "dlogits", "dW1", "db1", "dw2", "db2"):
        assert torch.equal(getattr(g1, f), getattr(g2, f)), f


def test_backward_layouts_agree():
    """NHWC and NCHW of the same layer give the same gradients (dx transposed)."""
    from paper_2608_23794_gb300 import moce
    cfg = LC("lay_nhwc", 2, 6, 10, 64, 24, 8, "f32", "nhwc", "relu", 64)
    g_h, ref_h, (lay, dev, dy, packed) = _run(cfg)
    xc = torch.from_numpy(synth.x_to_layout(lay.x, "nhwc", "nchw")).cuda()
    dyc = dy.permute(0, 3, 1, 2).contiguous()
    g_c = moce.moce_backward(xc, dyc, "nchw", packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"],
                             cfg.tau_min, cfg.tau_max)
    _close(g_c.dx.permute(0, 2, 3, 1).cpu().numpy(), ref_h["dx"], "dx nchw")
    _close(g_c.dlogits.cpu().numpy(), ref_h["dlogit"], "dlogits nchw")
    _close(g_c.dW1.cpu().numpy(), ref_h["dW1"], "dW1 nchw")


def test_backward_empty_batch_zeroes_parameter_gradients():
    from paper_2608_23794_gb300 import moce
    cfg = LC("empty", 0, 4, 4, 32, 8, 4, "f32", "nhwc", "relu", 32)
    lay = synth.make_layer(cfg.replace(N=1), seed=1)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    x = torch.empty((0, 4, 4, 32), device="cuda")
    dy = torch.empty((0, 4, 4, 9), device="cuda")
    g = moce.moce_backward(x, dy, "nhwc", packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"],
                           cfg.tau_min, cfg.tau_max)
    torch.cuda.synchronize()
    for f in ("dlogits", "dW1", "db1", "dw2", "db2"):
        assert float(getattr(g, f).abs().max()) == 0.0, f


def test_backward_dy_on_residual_only_reaches_unselected_channels():
    """With dy zero on every routed expert, dx is dy_res / |U| on U and 0 elsewhere,
    and every parameter gradient is zero (Eq. (res) has no parameters)."""
    from paper_2608_23794_gb300 import moce
    cfg = LC("res_only", 2, 7, 9, 96, 10, 6, "f32", "nhwc", "relu", 40)
    lay = synth.make_layer(cfg, seed=4)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    dyv, _ = synth.make_dy(cfg, seed=4)
    dyv[..., : cfg.C_out] = 0.0
    g = moce.moce_backward(dev["x"], torch.from_numpy(dyv).cuda(), "nhwc", packed, dev["W1"],
                           dev["b1"], dev["w2"], dev["b2"], cfg.tau_min, cfg.tau_max)
    _, _, resid = oracle_packed(lay)
    want = np.zeros(lay.x.shape, np.float32)
    want[..., resid] = (dyv[..., cfg.C_out] / len(resid))[..., None]
    np.testing.assert_allclose(g.dx.cpu().numpy(), want, rtol=1e-6, atol=0)
    for f in ("dlogits", "dW1", "db1", "dw2", "db2"):
        assert float(getattr(g, f).abs().max()) == 0.0, f


@pytest.mark.parametrize("cfg", [
    LC("k_eq_c_empty_u", 2, 3, 5, 12, 4, 12, "f32", "nhwc", "relu", 12),     # |U| = 0
    LC("one_expert", 3, 4, 4, 16, 1, 5, "f32", "nchw", "gelu", 16),          # R = 1
    LC("one_channel_k1", 2, 3, 3, 1, 3, 1, "f32", "nhwc", "relu", 1),        # C = k = 1
    LC("hw1_bf16", 5, 1, 1, 64, 7, 8, "bf16", "nhwc", "relu", 48),           # one position
], ids=lambda c: c.name)
def test_backward_degenerate_shapes(cfg):
    g, ref, _ = _run(cfg, seed=7)
    _close(g.dx.cpu().numpy(), ref["dx"], "dx")
    _close(g.dlogits.cpu().numpy(), ref["dlogit"], "dlogits")
    _close(g.dW1.cpu().numpy(), ref["dW1"], "dW1")
    _close(g.db1.cpu().numpy(), ref["db1"], "db1")
    _close(g.dw2.cpu().numpy(), ref["dw2"], "dw2")
    _close(g.db2.cpu().numpy(), np.array([ref["db2"]]), "db2")
