"""Failure detection on the GPU without a fault: a bounded device wait is
made to run out (a test hook gives the decode expert kernel's wait for a token
tile's gate/up results an unreachable target and a short budget). The kernel
gives up, lets its copies land, frees its tensor memory and returns; the
host reads ACE_ERR_TIMEOUT from the error word; the context stays usable and
the next forward passes replay parity."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import _replay as RP
import oracle as O
from paper_2609_05228_gb300 import ace, offline, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ace.lib()
    yield


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()


def _host(t):
    return (t.view(torch.int16).cpu().numpy().view(np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def test_bounded_wait_runs_out_and_is_reported():
    spec = synth.LayerSpec(256, 16, 4, 128, dtype="bf16")
    w = synth.make_layer(spec, seed=5)
    w.extra["a_gsp"], w.extra["a_rcr"] = offline.tables(w)
    layer = ace.AceLayer(w, w.extra["a_gsp"], w.extra["a_rcr"], max_tokens=64)
    T = 64
    x = synth.make_tokens(spec, T, seed=1)
    xd = _dev(x)
    out = torch.empty_like(xd)
    try:
        ace.ace_debug_set_wait_budget(layer.handle, 200_000)       # about 0.1 ms of SM clock
        layer.forward(xd, out, T, "ratio", 0.5)
        with pytest.raises(ace.AceError) as e:
            ace.ace_layer_sync(layer.handle)
        assert e.value.status == 5                                  # ACE_ERR_TIMEOUT
        ace.ace_layer_sync(layer.handle)                            # reported once: the word is cleared
    finally:
        ace.ace_debug_set_wait_budget(layer.handle, 0)
    # the context and the layer still work: a normal forward passes replay parity
    layer.forward(xd, out, T, "ratio", 0.5)
    ace.ace_layer_sync(layer.handle)
    dec, z = RP.replay_decision(layer.handle, spec, w.extra["a_gsp"], w.extra["a_rcr"], T, "ratio", 0.5)
    RP.check_logits(z, x, w)
    RP.compare(_host(out), O.moe_forward(x, w, decision=dec))
    with pytest.raises(ace.AceError):
        ace.ace_debug_set_wait_budget(layer.handle, -1)
    layer.close()
