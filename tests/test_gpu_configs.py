"""GPU parity on the remaining workload shapes, in replay mode (each
forward's own float32 logits through the oracle's float32 decision spec,
bit-exact; the fp64 oracle under that decision; every token compared):
* the 4-layer stack of the Qwen3-30B-A3B-shaped layer (distinct seeded
  weights per layer, residual x + y, skip ratio 0.5), prefill 16384 tokens
  and decode 32 tokens, layer by layer on the GPU's own bf16 intermediate
  activations;
* the large layer (hidden 4096, 256 experts, top-8, FFN 2048, Zipf routing),
  decode {1, 16, 128} and prefill {2048, 8192} tokens over the skip ratios
  0-0.625 in steps of 0.125: the decision over the whole batch, the outputs
  of every token up to 128 tokens and of a seeded 64-token sample above.
"""
import math

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


_STACK = {}


def _stack():
    if not _STACK:
        spec = synth.spec_qwen()
        ws, layers = [], []
        for l in range(4):
            w = synth.make_layer(spec, seed=100 + l)
            w.extra["a_gsp"], w.extra["a_rcr"] = offline.tables(w)
            ws.append(w)
            layers.append(ace.AceLayer(w, w.extra["a_gsp"], w.extra["a_rcr"], max_tokens=16384, residual=True))
        _STACK["w"], _STACK["layers"] = ws, layers
    return _STACK["w"], _STACK["layers"]


@pytest.mark.parametrize("T", [32, 16384])
def test_stack_of_four_layers(T):
    """Chained residual layers, layer by layer: each layer's decision replayed
    bit-exact from its own logits, and its output bf16(x_l + y_l) compared on
    every token with x_l + the oracle's y_l, where x_l is the GPU's own bf16
    input to that layer. The end of the stack is also compared with the
    oracle's independent fp64 stack (reported, boundary tokens differ)."""
    ws, layers = _stack()
    spec = ws[0].spec
    x0 = synth.make_tokens(spec, T, seed=1)
    cur = _dev(x0)
    for l, (w, layer) in enumerate(zip(ws, layers)):
        nxt = torch.empty_like(cur)
        layer.forward(cur, nxt, T, "ratio", 0.5)
        torch.cuda.synchronize()
        x_l = _host(cur)
        out_l = _host(nxt)
        dec, z_gpu = RP.replay_decision(layer.handle, spec, w.extra["a_gsp"], w.extra["a_rcr"], T, "ratio", 0.5)
        z_ref = RP.check_logits(z_gpu, x_l, w)
        y_ref = O.moe_forward(x_l, w, decision=dec)
        RP.compare_residual(out_l, x_l, y_ref, what=f"layer {l}")
        dec64 = O.ace_decide(z_ref, spec.top_k, w.extra["a_gsp"], w.extra["a_rcr"], "ratio", 0.5)
        RP.note_disagreement(f"stack T={T} layer {l}", dec, dec64)
        cur = nxt


_LARGE = {}


def _large():
    if not _LARGE:
        spec = synth.spec_large(zipf=True)
        w = synth.make_layer(spec, seed=0)
        # the GPU tables (checked against the oracle in test_large_layer_tables_device)
        w.extra["a_gsp"], w.extra["a_rcr"] = offline.tables_device(w)
        _LARGE["w"] = w
        _LARGE["layer"] = ace.AceLayer(w, w.extra["a_gsp"], w.extra["a_rcr"], max_tokens=8192)
    return _LARGE["w"], _LARGE["layer"]


LARGE_CASES = [(1, 0.0), (1, 0.5), (16, 0.0), (16, 0.125), (16, 0.25), (128, 0.25), (128, 0.375), (128, 0.5),
               (128, 0.625), (2048, 0.0), (2048, 0.125), (2048, 0.5), (8192, 0.0), (8192, 0.375), (8192, 0.5),
               (8192, 0.625)]


@pytest.mark.parametrize("T,q", LARGE_CASES)
def test_large_layer(T, q):
    w, layer = _large()
    spec = w.spec
    x = synth.make_tokens(spec, T, seed=1)
    xd = _dev(x)
    out = torch.empty_like(xd)
    layer.forward(xd, out, T, "ratio", q)
    torch.cuda.synchronize()
    y_gpu = _host(out)
    dec, z_gpu = RP.replay_decision(layer.handle, spec, w.extra["a_gsp"], w.extra["a_rcr"], T, "ratio", q)
    n_all = T * spec.top_k
    assert dec["count"] == min(O.llround_pos(float(np.float32(q)) * n_all), T * (spec.top_k - 1))
    sample = np.arange(T) if T <= 128 else np.sort(np.random.Generator(np.random.PCG64(7)).choice(T, 64, replace=False))
    z_ref = RP.check_logits(z_gpu, x, w, tokens=sample)
    y_ref = O.moe_forward(x, w, decision=dec, tokens=sample)
    RP.compare(y_gpu[sample], y_ref)
    if T <= 128:
        dec64 = O.ace_decide(z_ref, spec.top_k, w.extra["a_gsp"], w.extra["a_rcr"], "ratio", q)
        RP.note_disagreement(f"large T={T} q={q}", dec, dec64)


def test_large_layer_tables_device():
    """GPU tables of the large layer (256 experts in nine chunks of the tile
    budget, the last one ragged): A^GSP ratios of sampled experts against the
    oracle's direct fp64 products on those experts (the normalisation is one
    constant, so A[e] / A[e'] = a~_e / a~_e'), and the whole A^RCR table."""
    w, _ = _large()
    a, r = w.extra["a_gsp"], w.extra["a_rcr"]
    idx = [0, 31, 137, 255]
    sub = O.gsp_table(w.gamma, w.w_gate[idx], w.w_up[idx], w.w_down[idx], 0.0)
    np.testing.assert_allclose(a[idx] / a[idx[0]], sub / sub[0], rtol=3e-5)
    r_ref = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, w.spec.eps)
    np.testing.assert_allclose(r, r_ref, rtol=3e-5)


@pytest.mark.parametrize("T", [32, 300, 4096])
def test_stack_api_matches_chained_layers(T):
    """ace_stack_forward (the prefill path computes each next layer's RMSNorm
    inside the combine) gives the same bits as chaining the layers' forwards,
    and leaves each layer's decision readable."""
    ws, layers = _stack()
    spec = ws[0].spec
    x = _dev(synth.make_tokens(spec, T, seed=3))
    cur = x
    for layer in layers:
        nxt = torch.empty_like(cur)
        layer.forward(cur, nxt, T, "ratio", 0.5)
        cur = nxt
    torch.cuda.synchronize()
    want = cur.view(torch.int16).cpu().numpy()
    masks = [ace.ace_last_skip_mask(layer.handle, T, spec.top_k)[0].copy() for layer in layers]
    st = ace.ace_stack_create([layer.handle for layer in layers])
    try:
        out = torch.empty_like(x)
        for _ in range(2):
            ace.ace_stack_forward(st, x, out, T, "ratio", 0.5)
            torch.cuda.synchronize()
            assert (out.view(torch.int16).cpu().numpy() == want).all()
        for layer, m in zip(layers, masks):
            assert (ace.ace_last_skip_mask(layer.handle, T, spec.top_k)[0] == m).all()
        xp = x.cpu().pin_memory()
        op = torch.empty_like(xp).pin_memory()
        for _ in range(2):                                               # capture, then replay
            ace.ace_stack_forward_host(st, xp, op, T, "ratio", 0.5)
            assert (op.view(torch.int16).numpy() == want).all()
        with pytest.raises(ace.AceError):
            ace.ace_stack_forward(st, x, x, T, "ratio", 0.5)            # out aliases x
    finally:
        ace.ace_stack_destroy(st)
    with pytest.raises(ace.AceError):
        ace.ace_stack_create([layers[0].handle, layers[0].handle])      # the same layer twice
