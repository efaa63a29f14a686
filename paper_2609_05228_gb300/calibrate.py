"""Fixed skip thresholds from a calibration batch (App. B.1's quantile mapping).

The paper turns a target skip ratio q into a fixed threshold tau by taking,
over an unlabeled calibration pass, the score below which a fraction q of the
candidate slots fall. `calibrate_taus` runs that mapping on the GPU: it calls
the layer's forward in ratio mode on the calibration tokens for each q and
reads back the tau the library derived (the same App. B.1 rule it uses per
batch). The returned taus are then used in threshold mode on other batches.
"""
from __future__ import annotations

from . import ace


def calibrate_taus(layer: "ace.AceLayer", x_calib, T: int, qs, stream=None, fusion="max") -> dict:
    """{q: tau} for the layer from the device tokens x_calib [T, d] (under the
    given skip rule: tau is a threshold on that rule's score)."""
    import torch
    out = torch.empty_like(x_calib)
    taus = {}
    for q in qs:
        ace.ace_moe_forward(layer.handle, x_calib, out, T, "ratio", float(q), stream, fusion)
        _, _, _, tau, _ = ace.ace_last_skip_mask(layer.handle, T, layer.spec.top_k)
        taus[float(q)] = float(tau)
    return taus
