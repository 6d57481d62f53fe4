"""moce_forward_noalloc: the forward for callers that cannot allocate device memory.

Such callers (allocator or pool callbacks, loops that forbid allocation after
start-up, plugins whose framework owns every buffer) cannot provide a
workspace; this entry point uses a fixed scratch array inside the library.
Its output must match moce_forward on the same inputs and the CPU oracle, on
consecutive calls that reuse the shared array. This file is named to run last.
"""
import numpy as np
import pytest

from moce_cases import TOL, assert_close, device_tensors, oracle_forward
from paper_2608_23794_gb300 import synth

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

CASES = [
    synth.CONFIGS["rn50_stage1_reduce"].replace(N=8),           # stream kernel
    synth.CONFIGS["tiny_f32_nchw"],                             # multi-kernel path
    synth.LayerConfig("c72", 3, 9, 11, 72, 9, 5, "bf16", "nhwc", "gelu", 60),
]


@pytest.mark.parametrize("cfg", CASES, ids=lambda c: c.name)
def test_noalloc_matches_forward_on_two_calls(cfg):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23794_gb300 import build, moce
    build.build()
    lay = synth.make_layer(cfg, seed=21)
    dev = device_tensors(lay)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    args = (dev["W1"], dev["b1"], dev["w2"], dev["b2"], cfg.tau_min, cfg.tau_max)
    ref = moce.moce_forward(dev["x"], cfg.layout, packed, *args)
    ref = ref.float().cpu().numpy().astype(np.float64)
    tol = TOL[cfg.dtype]
    yref = oracle_forward(lay)
    for _ in range(2):
        got = moce.moce_forward_noalloc(dev["x"], cfg.layout, packed, *args)
        moce.moce_noalloc_check_device_error()
        got = got.float().cpu().numpy().astype(np.float64)
        assert np.all(np.abs(got - ref) <= tol + tol * np.abs(ref))
        assert_close(got, yref, cfg.dtype, "noalloc y")


def test_noalloc_rejects_layers_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23794_gb300 import build, moce
    build.build()
    cfg = synth.CONFIGS["rn50_stage3_reduce"]  # its workspace is well above 8 MiB
    assert moce.moce_workspace_bytes(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k) > (8 << 20)
    small = synth.make_layer(cfg.replace(N=1), seed=0)
    dev = device_tensors(small)
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    x = torch.zeros((cfg.N, cfg.H, cfg.W, cfg.C_in), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(moce.MoceError) as ei:
        moce.moce_forward_noalloc(x, "nhwc", packed, dev["W1"], dev["b1"], dev["w2"], dev["b2"],
                                  0.2, 6.0)
    assert ei.value.status == moce.MOCE_ERR_UNSUPPORTED
