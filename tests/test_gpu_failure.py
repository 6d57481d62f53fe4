"""Failure detection of the forward, without faulting the GPU.

The fault is made on the host: the workspace's fault-injection word
(control word 4) names work item 0, the first tile of example 0, whose
channel sums are then computed but never added to the example's
accumulator words. The stream kernel's gate for that example, and every
wait on its weights, then runs out its bounded wait. The forward must exit,
report MOCE_ERR_TIMEOUT through moce_check_device_error, leave the context
usable, and a re-initialised workspace must give correct results.
"""
import numpy as np
import pytest

from moce_cases import assert_close, device_tensors, oracle_forward
from paper_2608_23794_gb300 import synth

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.mark.parametrize("path", ["stream"])
def test_bounded_wait_reports_timeout_and_recovers(path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23794_gb300 import build, moce
    build.build()
    cfg = synth.LayerConfig("fail", 4, 16, 16, 64, 16, 4, "bf16", "nhwc", "relu", 56)
    lay = synth.make_layer(cfg, seed=9)
    dev = device_tensors(lay)
    assert moce.moce_forward_launches(dev["x"], "nhwc", cfg.C_out, cfg.k, path=path) == 1
    packed = moce.moce_pack_supports(dev["support_idx"], dev["support_logits"], cfg.C_in)
    ws = moce.Workspace(cfg.N, cfg.H, cfg.W, cfg.C_in, cfg.C_out, cfg.k)
    run = lambda: moce.moce_forward(dev["x"], "nhwc", packed, dev["W1"], dev["b1"], dev["w2"],
                                    dev["b2"], cfg.tau_min, cfg.tau_max, ws=ws, path=path)
    run()
    moce.moce_check_device_error(ws)

    ws.buffer[16:20].view(torch.int32).fill_(1)  # item 0 = POOL(0, 0) does not publish
    run()
    with pytest.raises(moce.MoceError) as ei:
        moce.moce_check_device_error(ws)
    assert ei.value.status == moce.MOCE_ERR_TIMEOUT

    ws.init()
    y = run()
    torch.cuda.synchronize()
    moce.moce_check_device_error(ws)
    assert_close(y.float().cpu().numpy().astype(np.float64), oracle_forward(lay), "bf16")
