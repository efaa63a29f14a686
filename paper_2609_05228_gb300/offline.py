"""Offline GSP and RCR tables (ACE Algorithms 2 and 3): host CPU, and GPU
(tables_device, through libace.so's ace_offline_tables_device).

The tables are computed once per layer from the frozen weights and handed to
ace_layer_create(). No calibration data is involved. The computation is the
host-only C++ library libace_offline.so (include/ace_offline.h: Gram-route
GSP, prototype-forward RCR, fp64, one expert per thread); this module is its
ctypes binding, with the C names.

Weights are nn.Linear-shaped: w_gate, w_up [N, m, d]; w_down [N, d, m];
bf16 arrays are uint16 bit patterns (passed as they are), others fp32.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import ace

LIBPATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "libace_offline.so")
_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        if not os.path.exists(LIBPATH):       # host-only C++: built on first use (g++, a few seconds)
            from . import build
            build.build_offline()
        L = ctypes.CDLL(LIBPATH)
        L.ace_offline_tables.restype = ctypes.c_int
        L.ace_offline_tables.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                         ctypes.c_void_p, ctypes.c_double, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_void_p, ctypes.c_void_p]
        _lib = L
    return _lib


def _host(a: np.ndarray, bf16: bool) -> np.ndarray:
    a = np.asarray(a)
    if bf16:
        if a.dtype != np.uint16:
            raise TypeError("bf16 weights are uint16 bit patterns")
        return np.ascontiguousarray(a)
    return np.ascontiguousarray(a, dtype=np.float32)


def ace_offline_tables(gamma, router_w, w_gate, w_up, w_down, eps: float = 1e-6, apply_gamma: bool = False,
                       n_threads: int = 0):
    """(A^GSP, A^RCR) float32 [N] from the layer's weights (see ace_offline.h)."""
    bf16 = np.asarray(w_gate).dtype == np.uint16
    n, m, d = np.asarray(w_gate).shape
    arrs = [_host(x, bf16) for x in (gamma, router_w, w_gate, w_up, w_down)]
    gsp = np.empty(n, np.float32)
    rcr = np.empty(n, np.float32)
    st = lib().ace_offline_tables(d, n, m, ace.ACE_BF16 if bf16 else ace.ACE_F32,
                                  *[x.ctypes.data for x in arrs], float(eps), int(bool(apply_gamma)),
                                  int(n_threads), gsp.ctypes.data, rcr.ctypes.data)
    if st != 0:
        raise ace.AceError(st, "ace_offline_tables failed")
    return gsp, rcr


def tables(layer, eps: float | None = None, apply_gamma: bool = False):
    """(A^GSP, A^RCR) as float32 arrays for a synth.LayerWeights-like layer."""
    e = layer.spec.eps if eps is None else eps
    return ace_offline_tables(layer.gamma, layer.router_w, layer.w_gate, layer.w_up, layer.w_down, e, apply_gamma)


def tables_device(layer, eps: float | None = None, apply_gamma: bool = False, device: int = 0,
                  tile_budget: int = 0):
    """(A^GSP, A^RCR) for a bf16 synth.LayerWeights-like layer, computed on the
    GPU by ace_offline_tables_device (libace.so); torch only holds the device
    copies of the weights for the call."""
    import torch

    if np.asarray(layer.w_gate).dtype != np.uint16:
        raise TypeError("the GPU tables take bf16 weights")
    dev = torch.device("cuda", device)

    def up(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)

    n, m, d = np.asarray(layer.w_gate).shape
    ts = [up(x) for x in (layer.gamma, layer.router_w, layer.w_gate, layer.w_up, layer.w_down)]
    torch.cuda.synchronize(dev)
    e = layer.spec.eps if eps is None else eps
    out = ace.ace_offline_tables_device(d, n, m, *ts, e, apply_gamma, tile_budget)
    del ts
    return out


def gsp_table(gamma, w_gate, w_up, w_down, eps: float = 1e-6) -> np.ndarray:
    """A^GSP alone (the router is not used by Algorithm 2)."""
    n, m, d = np.asarray(w_gate).shape
    bf16 = np.asarray(w_gate).dtype == np.uint16
    wr = np.zeros((n, d), np.uint16 if bf16 else np.float32)
    return ace_offline_tables(gamma, wr, w_gate, w_up, w_down, eps)[0]


def rcr_table(router_w, gamma, w_gate, w_up, w_down, eps: float = 1e-6, apply_gamma: bool = False) -> np.ndarray:
    """A^RCR alone."""
    return ace_offline_tables(gamma, router_w, w_gate, w_up, w_down, eps, apply_gamma)[1]
